// cci_gemm_ws_bf16.cu -- bf16 layers of the workspace family: the kernel
// configurations (activation source x N tile) and the choice among them.
#include "cci_gemm_ws.cuh"

namespace cci {

cudaError_t launch_gemm_ws_bf16(const FwdParams &p, cudaStream_t stream)
{
    using namespace ws;
    Plan pl;
    plan_layer(p, false, 64, &pl);
    const int asrc = pl.asrc;
    const int bn = choose_bn(m_tiles_of(p, asrc, pl.box), p.Cout, 256);
#define CCI_WS_CASE(A, N) \
    if (asrc == A && bn == N) return launch_cfg<false, A, N>(p, pl.box, pl.am, stream);
    CCI_WS_CASE(kA2d, 64)
    CCI_WS_CASE(kA2d, 128)
    CCI_WS_CASE(kA2d, 256)
    CCI_WS_CASE(kA4d, 64)
    CCI_WS_CASE(kA4d, 128)
    CCI_WS_CASE(kA4d, 256)
    CCI_WS_CASE(kAGather, 64)
    CCI_WS_CASE(kAGather, 128)
    CCI_WS_CASE(kAGather, 256)
#undef CCI_WS_CASE
    return cudaErrorInvalidValue;
}

}  // namespace cci
