// cci_gemm_pk.cu -- the fused tensor-core family (CCI_ALGO_DENSE_TC): the GEMM
// of the workspace family with the packed weights expanded into each B tile by
// the producer warps (no workspace, no decompression launch).  Single-CTA tiles
// (N tile 64 or 128); the CTA-pair tiles are in cci_gemm_pk_pair.cu.
#include "cci_gemm_ws.cuh"

namespace cci {

cudaError_t launch_gemm_pk_pair(const FwdParams &p, int asrc, const ws::Plan &pl, cudaStream_t stream);

// conditions of the packed-weight copies and of the expansion: G in
// {4, 8, 16, 32}, K in {1, 2, 4, 8} with K <= G / 2, R * K % 16 == 0 (16-byte
// rows of the packed arrays), R * K < 2^31 (copy coordinates), 16-byte aligned
// packed arrays
bool gemm_pk_shape_ok(const FwdParams &p)
{
    const bool gk = (p.G == 4 || p.G == 8 || p.G == 16 || p.G == 32) &&
                    (p.K == 1 || p.K == 2 || p.K == 4 || p.K == 8) && 2 * p.K <= p.G;
    if (!gk) return false;
    if ((p.R * p.K) % 16 != 0 || p.R * p.K >= (int64_t(1) << 31)) return false;
    return reinterpret_cast<uintptr_t>(p.values) % 16 == 0 && reinterpret_cast<uintptr_t>(p.idx) % 16 == 0;
}

// ... and activations the GEMM copies by TMA (not the row gather)
bool gemm_pk_supported(const FwdParams &p)
{
    if (!gemm_pk_shape_ok(p)) return false;
    ws::Plan pl;
    ws::plan_layer(p, false, 64, &pl);
    return pl.asrc != ws::kAGather;
}

cudaError_t launch_gemm_pk(const FwdParams &p, cudaStream_t stream)
{
    using namespace ws;
    if (!gemm_pk_shape_ok(p)) return cudaErrorNotSupported;
    Plan pl;
    plan_layer(p, false, 64, &pl);
    const int asrc = pl.asrc;
    if (asrc == kAGather) return cudaErrorNotSupported;
    const int64_t m_tiles = m_tiles_of(p, asrc, pl.box);
    const int64_t nks = (p.R + 63) / 64;
    // CTA pairs on long reductions with 256-wide N tiles, as the workspace family
    if ((asrc == kA2d || asrc == kA4d) && nks >= 16 && choose_bn(m_tiles, p.Cout, 256, 2) == 256)
        return launch_gemm_pk_pair(p, asrc, pl, stream);
    // one producer item per thread: B tiles of at most 128 rows per CTA
    const int bn = choose_bn(m_tiles, p.Cout, 128, 1);
#define CCI_PK_CASE(A, N) \
    if (asrc == A && bn == N) return launch_cfg<false, A, N, 1, 1, true>(p, pl.box, pl.am, stream);
    CCI_PK_CASE(kA2d, 64)
    CCI_PK_CASE(kA2d, 128)
    CCI_PK_CASE(kA4d, 64)
    CCI_PK_CASE(kA4d, 128)
    CCI_PK_CASE(kAHalo, 64)
    CCI_PK_CASE(kAHalo, 128)
#undef CCI_PK_CASE
    return cudaErrorInvalidValue;
}

}  // namespace cci
