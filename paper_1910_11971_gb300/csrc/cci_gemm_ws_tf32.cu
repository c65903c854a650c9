// cci_gemm_ws_tf32.cu -- fp32 layers of the workspace family (the split product:
// tf32 hi*hi plus bf16 cross terms): the kernel configurations and the choice
// among them.
#include "cci_gemm_ws.cuh"

namespace cci {

cudaError_t launch_gemm_ws_tf32(const FwdParams &p, cudaStream_t stream)
{
    using namespace ws;
    Plan pl;
    plan_layer(p, true, 32, &pl);
    const int asrc = pl.asrc;
    const int bn = choose_bn(m_tiles_of(p, asrc, pl.box), p.Cout, 128);
    // TMA-copied activations: clusters of two CTAs on adjacent M tiles share each
    // weight tile by multicast (half the weight copies per CTA)
#define CCI_WS_MC(A, N) \
    if (asrc == A && bn == N) return launch_cfg<true, A, N, 1, 1, false, true>(p, pl.box, pl.am, stream);
    CCI_WS_MC(kA2d, 64)
    CCI_WS_MC(kA2d, 128)
    CCI_WS_MC(kA4d, 64)
    CCI_WS_MC(kA4d, 128)
#undef CCI_WS_MC
#define CCI_WS_CASE(A, N) \
    if (asrc == A && bn == N) return launch_cfg<true, A, N, 1>(p, pl.box, pl.am, stream);
    CCI_WS_CASE(kAGather, 64)
    CCI_WS_CASE(kAGather, 128)
#undef CCI_WS_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_ws(const FwdParams &p, int dtype, cudaStream_t stream)
{
    return dtype == CCI_F32 ? launch_gemm_ws_tf32(p, stream) : launch_gemm_ws_bf16(p, stream);
}

}  // namespace cci
