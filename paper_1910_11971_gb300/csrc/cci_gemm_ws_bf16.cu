// cci_gemm_ws_bf16.cu -- bf16 layers of the workspace family: the kernel
// configurations (activation source x N tile x CTAs per tile) and the choice
// among them.
#include "cci_gemm_ws.cuh"

namespace cci {

cudaError_t launch_gemm_ws_bf16(const FwdParams &p, cudaStream_t stream)
{
    using namespace ws;
    Plan pl;
    plan_layer(p, false, 64, &pl);
    const int asrc = pl.asrc;
    // products of fewer than 64 reduction indices copy only those (stage_k_in)
    const int kin = stage_k_in(p, false, asrc, false);
    if (kin < 64 && !build_a_maps(p, pl.box, asrc, false, kin, &pl.am)) return cudaErrorInvalidValue;
    const int64_t m_tiles = m_tiles_of(p, asrc, pl.box);
    const int64_t nks = (p.R + 63) / 64;
    // CTA pairs (256-row tiles, B split over the pair) halve each SM's B traffic,
    // which pays on long reductions with 256-wide N tiles; shorter or narrower
    // layers run faster on single CTAs (measured on the ResNet-50 stack)
    const bool pair = (asrc == kA2d || asrc == kA4d) && nks >= 16 && choose_bn(m_tiles, p.Cout, 256, 2) == 256;
    if (pair) {
        if (asrc == kA2d) return launch_cfg<false, kA2d, 256, 2>(p, pl.box, pl.am, stream);
        return launch_cfg<false, kA4d, 256, 2>(p, pl.box, pl.am, stream);
    }
    const int bn = choose_bn(m_tiles, p.Cout, 256, 1);
    if (asrc == kAHalo) {
        // 3x3 convolutions from halo copies (tiles of nine stages per chunk at least)
        // CTA pairs (256-row tiles, each CTA copying its own halo and half of every
        // weight tile) for layers of 256+ input channels whose 256-wide N tile wins
        // the pair tile-round count: every tile re-reads the layer's weights, whose
        // copies bound those layers (14 x 14 ResNet-50 layers: 0.0396 -> 0.0375 ms)
        if (p.Cin >= 256 && choose_bn(m_tiles, p.Cout, 256, 2) == 256)
            return launch_cfg<false, kAHalo, 256, 2>(p, pl.box, pl.am, stream);
        if (bn == 64) return launch_cfg<false, kAHalo, 64, 1>(p, pl.box, pl.am, stream);
        if (bn == 128) return launch_cfg<false, kAHalo, 128, 1>(p, pl.box, pl.am, stream);
        return launch_cfg<false, kAHalo, 256, 1>(p, pl.box, pl.am, stream);
    }
    // tiles of at most 4 stages: the output write dominates, two epilogue groups
    // with two staging buffers each; longer ones keep the shared memory for stages
    const bool short_k = nks <= 4 && asrc != kAGather;
    if (short_k) {
#define CCI_WS_SHORT(A, N) \
    if (asrc == A && bn == N) return launch_cfg<false, A, N, 1, 2>(p, pl.box, pl.am, stream);
        CCI_WS_SHORT(kA2d, 64)
        CCI_WS_SHORT(kA2d, 128)
        CCI_WS_SHORT(kA2d, 256)
        CCI_WS_SHORT(kA4d, 64)
        CCI_WS_SHORT(kA4d, 128)
        CCI_WS_SHORT(kA4d, 256)
#undef CCI_WS_SHORT
    }
#define CCI_WS_CASE(A, N) \
    if (asrc == A && bn == N) return launch_cfg<false, A, N, 1>(p, pl.box, pl.am, stream);
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
