// cci_gemm_pk_pair.cu -- CTA-pair tiles of the fused tensor-core family
// (256 x 256 over two SMs, tcgen05.mma cta_group::2): each CTA expands the
// packed weights of its 128 B rows; the odd CTA's producers release their
// writes to the even CTA's full barrier.
#include "cci_gemm_ws.cuh"

namespace cci {

cudaError_t launch_gemm_pk_pair(const FwdParams &p, int asrc, const ws::Plan &pl, cudaStream_t stream)
{
    using namespace ws;
    if (asrc == kA2d) return launch_cfg<false, kA2d, 256, 2, 1, true>(p, pl.box, pl.am, stream);
    if (asrc == kA4d) return launch_cfg<false, kA4d, 256, 2, 1, true>(p, pl.box, pl.am, stream);
    return cudaErrorInvalidValue;
}

}  // namespace cci
