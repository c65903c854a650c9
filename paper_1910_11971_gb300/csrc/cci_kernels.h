// cci_kernels.h -- launchers shared between the libcci translation units.
#pragma once

#include "cci_common.cuh"

namespace cci {

cudaError_t launch_pack(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                        uint8_t *idx, uint32_t *status, cudaStream_t stream);
cudaError_t launch_td_mask(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, float rate,
                           const float *u, void *Wout, uint8_t *mask, uint32_t *status, cudaStream_t stream);
// balanced sparsity, the comparison format (cci_bbs.cu)
cudaError_t launch_bbs_pack(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                            uint8_t *idx, uint32_t *status, cudaStream_t stream);
cudaError_t launch_bbs_decompress(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream);
cudaError_t launch_bbs_gather(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream);
cudaError_t launch_pack_stats(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K,
                              unsigned long long *counts, cudaStream_t stream);
cudaError_t launch_generic(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream);
cudaError_t launch_fma_probe(float *out, int blocks, int threads, int iters, cudaStream_t stream);
// bounded-wait diagnostic (cci_dense_tc.cu): arrive = 0 lets the wait expire
cudaError_t launch_wait_probe(uint32_t *status, int arrive, cudaStream_t stream);

// (G, K) pairs of the workspace tensor-core family
bool dense_tc_supported(int dtype, int G, int K);
// decompress once into p.wdense and copy B tiles from it (bf16: dense [Cout][R];
// fp32: the two operand planes of the split, cci_common.cuh)
cudaError_t launch_dense_tc_ws(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream);
// dense fp32 W[Cout][R] (R % 4 == 0, 16-byte aligned) into the operand planes at planes
cudaError_t launch_dense_split(const uint32_t *W, int64_t Cout, int64_t R, void *planes, cudaStream_t stream);

// dense product on the tensor cores from the decompressed workspace p.wdense
// (cci_gemm_ws_*.cu): bf16 dense [Cout][R], or the fp32 operand planes
cudaError_t launch_gemm_ws(const FwdParams &p, int dtype, cudaStream_t stream);
cudaError_t launch_gemm_ws_bf16(const FwdParams &p, cudaStream_t stream);
cudaError_t launch_gemm_ws_tf32(const FwdParams &p, cudaStream_t stream);

// fused tensor-core product (cci_gemm_pk*.cu): the GEMM of the workspace family
// with the packed weights (p.values, p.idx, p.G, p.K) expanded into each B tile
// in shared memory; bf16 only.  gemm_pk_shape_ok: (G, K), packed-array shape and
// alignment allow it; gemm_pk_supported: also the activations are copied by
// TMA; launch_gemm_pk returns cudaErrorNotSupported, before any launch, for a
// layer without it.
bool gemm_pk_shape_ok(const FwdParams &p);
bool gemm_pk_supported(const FwdParams &p);
cudaError_t launch_gemm_pk(const FwdParams &p, cudaStream_t stream);

// One register-tiled instantiation: (dtype, G, K) -> tile shape and launcher.
struct RegtileEntry {
    int dtype, G, K, MG, T, D;
    const char *name;
    cudaError_t (*launch)(const FwdParams &p, cudaStream_t stream);
};

// all instantiations, terminated by an entry with launch == nullptr
const RegtileEntry *regtile_table();

// channel-warps per CTA (4 or 8) for a layer with this many groups
int regtile_wc(int64_t groups, int MG);

constexpr size_t kMaxSmemPerBlock = 227 * 1024;

}  // namespace cci
