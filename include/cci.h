/*
 * cci.h -- C ABI of libcci.so: forward products of layers with cross-channel
 * intragroup (CCI) sparsity on NVIDIA GB300 (sm_103a).
 *
 * Method: Yu et al., "Cross-Channel Intragroup Sparsity Neural Network"
 * (arXiv 1910.11971).  For every input feature r of a layer (for a convolution,
 * every tap (kh, kw, ci)), the weights of G neighbouring output channels form a
 * group, and exactly K of the G are kept (Sec. 3.1, Fig. 1).  Every G rows of the
 * weight matrix therefore compress into K rows of (value, index) pairs, each with
 * as many columns as the original matrix; the index is the plain row index
 * inside the group (log2 G bits, Sec. 3.1).  The product H = W x X is then Alg. 2
 * of Sec. 3.2: H(G*i + Idx, j) += Val * X(k, j).
 *
 * Layouts (all row-major, dense, contiguous; element = dtype unless stated):
 *   W       [Cout][R]              dense weights (pack input); R = Cin*KH*KW,
 *                                  r = (kh*KW + kw)*Cin + ci for convolutions
 *                                  (OHWI order)
 *   values  [Cout/G][R][K]         kept weights, per (group, r) in increasing index
 *   idx     [Cout/G][R][K] uint8   index j in [0, G) of each kept weight
 *   X       [N][Cin]               product input: N columns of Cin features
 *                                  (the paper's column-major X)
 *   X       [B][H][W][Cin]         convolution input (NHWC)
 *   Y       [N][Cout] float32      product output (the paper's H, transposed)
 *   Y       [B][P][Q][Cout] float32  convolution output (NHWC),
 *                                  P = (H + 2*pad_h - KH)/stride_h + 1, Q likewise
 *
 * Ownership and execution: the caller allocates every buffer; all data pointers
 * are DEVICE pointers (except the X_host / Y_host of cci_linear_host); the
 * library allocates nothing.  It keeps no state between calls except two
 * per-device caches, both filled on a device's first use: the dynamic
 * shared-memory limit set on each tensor-core kernel, and the device address of
 * the static scratch array of cci_linear_dense_tc_static (see there).  Every
 * call is asynchronous on `stream` (NULL = the legacy default stream) and
 * returns once its kernels are enqueued.  Calls on different streams may run
 * concurrently when their outputs do not overlap.
 *
 * Errors:
 *   - Argument errors are detected on the host, before anything is enqueued, and
 *     returned directly (nothing is written).
 *   - A failed launch returns CCI_ERR_CUDA.
 *   - Errors found by the kernels while they run (NaN in a pack input, a packed
 *     index >= G, an expired bounded wait) are OR-ed as bits (1u << code) into
 *     the caller's device word `*dev_status`, if it is not NULL; read it after
 *     synchronising the stream and decode it with cci_decode_device_status().
 *     The library never clears that word.  When a kernel reports an error its
 *     outputs are unspecified.
 */
#ifndef CCI_H_
#define CCI_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* the same type as cudaStream_t */
typedef struct CUstream_st *cci_stream_t;

typedef enum cci_status {
    CCI_OK = 0,
    CCI_ERR_NULL = 1,         /* a required pointer is NULL */
    CCI_ERR_SHAPE = 2,        /* a size is negative/zero where not allowed, too large,
                                 or the convolution geometry has no output */
    CCI_ERR_GROUP = 3,        /* G not in [1, 256], K not in [1, G], or Cout % G != 0 */
    CCI_ERR_DTYPE = 4,        /* dtype is not a cci_dtype */
    CCI_ERR_ALIGN = 5,        /* a pointer is not aligned to its element size */
    CCI_ERR_VALUE = 6,        /* device: NaN among the weights given to cci_pack */
    CCI_ERR_CUDA = 7,         /* a CUDA launch or runtime call failed */
    CCI_ERR_TIMEOUT = 8,      /* device: a bounded wait inside a kernel expired */
    CCI_ERR_UNSUPPORTED = 9,  /* valid request this build does not implement */
    CCI_ERR_INDEX = 10,       /* device: a packed index >= G given to a product (dense
                                 kernels: also an index set not strictly increasing) */
    CCI_ERR_WORKSPACE = 11    /* the kernel family needs a workspace: missing, too small
                                 or not 16-byte aligned (see cci_workspace_size) */
} cci_status;

typedef enum cci_dtype {
    CCI_F32 = 0,   /* IEEE binary32 */
    CCI_BF16 = 1   /* bfloat16; products accumulate in fp32 on the exact values */
} cci_dtype;

/* Kernel family for cci_linear_ex / cci_conv2d_ex. */
typedef enum cci_algo {
    CCI_ALGO_AUTO = 0,      /* the fastest family this build has for (G, K, dtype, shape): the
                               workspace tensor-core family when a large enough workspace is
                               given (cci_linear_ws); else the fused tensor-core family
                               (CCI_ALGO_DENSE_TC) for bf16 layers that have it; else the
                               CUDA-core families */
    CCI_ALGO_GENERIC = 1,   /* generic kernel: any G <= 256, any K, any alignment */
    CCI_ALGO_REGTILE = 2,   /* register-tiled scatter on CUDA cores: Alg. 2 with the output
                               row chosen per (group, r) by a warp-uniform jump;
                               CCI_ERR_UNSUPPORTED when (G, K, dtype, shape) has no tile */
    CCI_ALGO_DENSE_TC = 3,  /* fused tensor-core family, no workspace: inside the GEMM the
                               packed (value, index) runs of each stage are copied by TMA
                               and expanded by producer warps into the dense bf16 weight
                               tile in shared memory (each value to row G*i + Idx of its
                               group, Alg. 2), which tcgen05.mma multiplies with the TMA-
                               copied activations.  bf16; G in {4, 8, 16, 32}, K in
                               {1, 2, 4, 8} with K <= G/2; Cin % 8 == 0, R*K % 16 == 0;
                               16-byte aligned X, Y, values and idx; activations a product
                               or a convolution with strides <= 2 and Cin % 64 == 0 (else
                               CCI_ERR_UNSUPPORTED).  Index sets are checked (strictly
                               increasing, < G; CCI_ERR_INDEX) by the CTAs of the first
                               column tile of every channel tile */
    CCI_ALGO_EXPAND = 4,    /* register-tiled on CUDA cores without jumps: each (group, r)
                               is expanded to its G weights (pruned ones zero) in shared
                               memory and all G rows are updated; same shape rules as
                               CCI_ALGO_REGTILE */
    CCI_ALGO_DENSE_TC_WS = 5  /* decompress the packed weights once per call into a caller
                               workspace and multiply densely on the tensor cores (tcgen05),
                               operands copied by TMA (cp.async.bulk.tensor).  bf16: dense bf16 [Cout][R],
                               Cin % 8 == 0, R % 8 == 0.  fp32: every operand split as
                               hi + lo (hi a tf32 value) and, per 32 indices, the product
                               hi(x) hi(w) on tf32 MMAs plus bf16(x) bf16(lo(w)) +
                               bf16(lo(x)) bf16(hi(w)) on bf16 MMAs (8 MMAs; per term
                               |error| <= 5.7e-6 |w||x| before the fp32 accumulation);
                               workspace: plane 0 [Cout][R] fp32 hi, then plane 1
                               [Cout][ceil(R/32)*64] bf16 (per 32-wide chunk of r, 32
                               bf16(hi(w)) then 32 bf16(lo(w))).  Cin % 4 == 0, R % 4 == 0.
                               Needs cci_workspace_size() bytes */
} cci_algo;

/*
 * cci_pack -- choose and compress the kept weights (Sec. 3.1 format, Sec. 5.1
 * selection: the weights of largest |w| survive).
 *
 * For every group gi in [0, Cout/G) and r in [0, R), the G weights
 * W[gi*G + j][r], j = 0..G-1, are ranked by decreasing |w| (compared in the
 * storage dtype; -0 and +0 are equal, +-inf is largest); equal magnitudes rank by
 * increasing j.  The first K survive and are written in increasing j:
 * values[gi][r][s] = W[gi*G + j_s][r] (bit-exact copy), idx[gi][r][s] = j_s.
 *
 *   W          device, [Cout][R] of dtype, aligned to the element size
 *   values     device, [Cout/G][R][K] of dtype (written)
 *   idx        device, [Cout/G][R][K] uint8 (written)
 *   dev_status device uint32 or NULL; NaN in W sets bit (1u << CCI_ERR_VALUE)
 *              (with NULL, NaN goes unreported and ranks above +inf)
 * Errors: CCI_ERR_NULL, CCI_ERR_SHAPE (Cout or R < 1), CCI_ERR_GROUP,
 *         CCI_ERR_DTYPE, CCI_ERR_ALIGN, CCI_ERR_CUDA.
 */
cci_status cci_pack(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K,
                    void *values, uint8_t *idx, uint32_t *dev_status, cci_stream_t stream);

/*
 * cci_linear -- Y = X W-hat^T for a CCI-sparse fully connected layer (Alg. 2 of
 * Sec. 3.2 over all N columns, with the slot loop for K > 1):
 *   Y[n][gi*G + idx[gi][r][s]] += values[gi][r][s] * X[n][r]
 * summed over r and s in fp32, starting from zero.  A repeated index inside one
 * (group, r) adds both values, as Alg. 2 does.
 *
 *   X          device, [N][Cin] of dtype (R = Cin)
 *   values,idx device, as written by cci_pack for (Cout, R = Cin, G, K)
 *   Y          device, [N][Cout] float32 (written, every element)
 *   dev_status device uint32 or NULL; an index >= G sets bit (1u << CCI_ERR_INDEX)
 * N = 0 is valid and enqueues nothing.
 * Errors: CCI_ERR_NULL, CCI_ERR_SHAPE, CCI_ERR_GROUP, CCI_ERR_DTYPE, CCI_ERR_ALIGN,
 *         CCI_ERR_CUDA.
 */
cci_status cci_linear(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                      const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                      float *Y, uint32_t *dev_status, cci_stream_t stream);

/*
 * cci_conv2d -- CCI-sparse 2-D convolution (Sec. 3.1: the structure applies to
 * convolutional layers with one group per tap (kh, kw, ci)), computed as an
 * implicit product: column n = (b, p, q), reduction index
 * r = (kh*KW + kw)*Cin + ci, and
 *   x[n][r] = X[b][p*stride_h - pad_h + kh][q*stride_w - pad_w + kw][ci]
 * or 0 outside the image (cross-correlation, zero padding, floor output size, no
 * dilation, conv groups or bias).
 *
 *   X          device NHWC [B][H][W][Cin] of dtype
 *   values,idx device, cci_pack output for W[Cout][KH*KW*Cin] (OHWI)
 *   Y          device NHWC [B][P][Q][Cout] float32 (written, every element)
 * B = 0 is valid and enqueues nothing.
 * Errors: as cci_linear; CCI_ERR_SHAPE also when P or Q < 1.
 */
cci_status cci_conv2d(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W,
                      int64_t Cin, const void *values, const uint8_t *idx, int64_t Cout,
                      int KH, int KW, int stride_h, int stride_w, int pad_h, int pad_w, int G,
                      int K, float *Y, uint32_t *dev_status, cci_stream_t stream);

/* As cci_linear / cci_conv2d, with the kernel family chosen by `algo` and no
 * workspace (CCI_ALGO_DENSE_TC_WS returns CCI_ERR_WORKSPACE; AUTO does not pick it,
 * but does pick the fused tensor-core family, which needs none). */
cci_status cci_linear_ex(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                         const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                         float *Y, uint32_t *dev_status, cci_algo algo, cci_stream_t stream);
cci_status cci_conv2d_ex(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W,
                         int64_t Cin, const void *values, const uint8_t *idx, int64_t Cout,
                         int KH, int KW, int stride_h, int stride_w, int pad_h, int pad_w,
                         int G, int K, float *Y, uint32_t *dev_status, cci_algo algo,
                         cci_stream_t stream);

/*
 * cci_workspace_size -- bytes of device workspace that cci_linear_ws /
 * cci_conv2d_ws need for this kernel family and layer (R = Cin for a product,
 * Cin*KH*KW for a convolution): for CCI_ALGO_DENSE_TC_WS Cout*R*2 (bf16) or
 * Cout*(R*4 + ceil(R/32)*128) (fp32: Cout*R*8 when R % 32 == 0), 0 for the
 * families that need none.  For CCI_ALGO_AUTO: the
 * bytes that let AUTO pick its fastest family (the dense tensor-core one).
 */
size_t cci_workspace_size(cci_algo algo, cci_dtype dtype, int64_t Cout, int64_t R);

/*
 * As cci_linear_ex / cci_conv2d_ex with a caller workspace (device, 16-byte
 * aligned, `workspace_bytes` long; NULL / 0 allowed for families that need
 * none).  The call overwrites the workspace; calls that overlap on the GPU must
 * use different workspaces.  CCI_ALGO_AUTO uses the dense tensor-core family
 * when the layer has one and the workspace is large enough, else the CUDA-core
 * family.
 */
cci_status cci_linear_ws(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                         const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                         float *Y, uint32_t *dev_status, cci_algo algo, void *workspace,
                         size_t workspace_bytes, cci_stream_t stream);
cci_status cci_conv2d_ws(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W,
                         int64_t Cin, const void *values, const uint8_t *idx, int64_t Cout,
                         int KH, int KW, int stride_h, int stride_w, int pad_h, int pad_w,
                         int G, int K, float *Y, uint32_t *dev_status, cci_algo algo,
                         void *workspace, size_t workspace_bytes, cci_stream_t stream);

/*
 * cci_linear_host -- the product H = W-hat x X of Alg. 2 (Sec. 3.2) with the
 * activations and the output in HOST memory: Y_host[N][Cout] (fp32) =
 * X_host[N][Cin] * Wd^T, Wd the dense matrix of the packed weights (which stay
 * on the device).  The columns are processed in chunks of `chunk_cols`; chunk c
 * is copied in on `copy_in_stream`, multiplied on `stream` (the dense
 * tensor-core family AUTO picks: the fused one from the packed weights, else the
 * workspace one, the weights decompressed once by the first chunk) and copied
 * out on `copy_out_stream`, so that the copies of neighbouring chunks overlap
 * the product.  The result equals cci_linear_ws with CCI_ALGO_AUTO and a
 * workspace on the same data bit for bit.
 *
 *   X_host, Y_host  host memory; page-locked (cudaHostAlloc / registered) for the
 *                   copies to overlap; pageable memory is correct but serialises
 *   values, idx     device, as cci_linear
 *   chunk_cols      columns per chunk, >= 1 (a multiple of 128 keeps the
 *                   product's tiles full)
 *   device_buffer   device, 256-byte aligned, at least
 *                   cci_linear_host_buffer_size(dtype, Cin, Cout, chunk_cols)
 *                   bytes: the workspace and two staging slots per direction;
 *                   overwritten
 *   copy_in_stream, copy_out_stream  may be NULL: that copy then runs on `stream`
 * Ordering: the copies start after the work enqueued on `stream` before the
 * call; `stream` waits for the last copy-out, so Y_host is complete once `stream`
 * has reached the end of the call's work (synchronise `stream` before reading
 * it).  Calls that overlap on the GPU must use different device buffers.
 * Errors: as cci_linear; CCI_ERR_SHAPE for chunk_cols < 1; CCI_ERR_UNSUPPORTED
 * for layers without the dense tensor-core kernel (it needs Cin % 4 == 0 for
 * fp32, % 8 for bf16, and G in {4, 8, 16, 32} with K <= G/2); CCI_ERR_WORKSPACE for a missing,
 * short or misaligned device buffer; CCI_ERR_CUDA if an event, copy or launch
 * fails (chunks already enqueued still complete on the streams).
 */
size_t cci_linear_host_buffer_size(cci_dtype dtype, int64_t Cin, int64_t Cout, int64_t chunk_cols);
cci_status cci_linear_host(const void *X_host, cci_dtype dtype, int64_t N, int64_t Cin,
                           const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                           float *Y_host, int64_t chunk_cols, void *device_buffer,
                           size_t device_buffer_bytes, uint32_t *dev_status, cci_stream_t stream,
                           cci_stream_t copy_in_stream, cci_stream_t copy_out_stream);

/*
 * cci_td_mask -- one step of the improved targeted dropout used to train CCI
 * layers (Sec. 5.1).  Per group of G output channels at one input index r the K
 * weights of largest |w| (those cci_pack keeps: same ranking, ties to the lower
 * index) are protected; each other weight is a pruning candidate and is dropped
 * for this training pass when its uniform draw is below `rate`:
 *   W_out[co][r] = 0 if (co is a candidate and uniforms[co][r] < rate) else W[co][r]
 *   mask[co][r]  = 1 if W_out keeps the weight, else 0      (mask may be NULL)
 * The paper starts the candidate drop rate at 0.5 and raises it toward 1 during
 * training (rate is the caller's schedule).  The random numbers are an input:
 * uniforms[Cout][R] fp32 in [0, 1), device.  W, W_out: device [Cout][R] of dtype
 * (W_out may not alias W); mask: device uint8 [Cout][R].  rate outside [0, 1]
 * or NaN: CCI_ERR_VALUE; NaN weights are reported in dev_status as for cci_pack;
 * other argument errors as for cci_pack.
 */
cci_status cci_td_mask(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K, float rate,
                       const float *uniforms, void *W_out, uint8_t *mask, uint32_t *dev_status,
                       cci_stream_t stream);

/*
 * cci_td_drop_rate -- the candidate drop rate of the targeted-dropout schedule
 * (Sec. 5.1) at training step `step`: the paper fixes only the end points (start
 * at 50 %, end toward 100 %); this library ramps linearly from `start` to `end`
 * over `ramp_steps` steps and holds `end` afterwards (ramp_steps <= 0: `end` at
 * once; negative steps count as 0).  Host function, no device work.
 */
float cci_td_drop_rate(int64_t step, int64_t ramp_steps, float start, float end);

/*
 * Balanced sparsity (Sec. 3.4), the format the paper compares CCI with: groups
 * run along the INPUT dimension.  Per output channel co and group of G
 * consecutive inputs r in [g*G, g*G + G) (R % G == 0), K weights are kept.
 *
 * cci_bbs_pack -- values[Cout][R/G][K] (dtype) and idx[Cout][R/G][K] (uint8,
 * offsets inside the group): the K of largest |w| per group, ties to the lower
 * index, in increasing index (the selection rule of cci_pack).  Errors as for
 * cci_pack; R % G != 0 is CCI_ERR_GROUP.
 *
 * cci_bbs_linear -- Y[N][Cout] fp32 = sum over groups and slots of
 * values[co][g][k] * X[n][g*G + idx[co][g][k]] (the gather form of the product).
 * algo CCI_ALGO_DENSE_TC_WS: decompression into the workspace and the tensor-core
 * product of the CCI path (Cin % 8 bf16 / % 4 fp32, Cout % 4, 16-byte aligned X,
 * Y and workspace of cci_workspace_size(CCI_ALGO_DENSE_TC_WS, dtype, Cout, Cin)
 * bytes); CCI_ALGO_GENERIC: the CUDA-core gather kernel (32 % G == 0); AUTO: the
 * first when the layer and workspace allow, else the second; other families:
 * CCI_ERR_UNSUPPORTED.  Index sets must be strictly increasing and < G
 * (CCI_ERR_INDEX in dev_status).  Everything else as for cci_linear_ws.
 */
cci_status cci_bbs_pack(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                        uint8_t *idx, uint32_t *dev_status, cci_stream_t stream);
cci_status cci_bbs_linear(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                          const uint8_t *idx, int64_t Cout, int G, int K, float *Y, uint32_t *dev_status,
                          cci_algo algo, void *workspace, size_t workspace_bytes, cci_stream_t stream);

/*
 * cci_pack_stats -- the allocation error of packing W (Sec. 4, Eq. 1, measured):
 * adds to counts[0] the number of nonzero weights of W[Cout][R] and to counts[1]
 * the number of them that cci_pack with (G, K) cannot keep (per group of G
 * output channels at one input index, the nonzeros beyond K).  counts[1] /
 * counts[0] estimates Eq. 1's P_d when the zeros of W are independent with
 * probability Ps and K = G*(1 - Ps).  A weight is nonzero when its magnitude
 * bits are (-0 counts as zero).  W: device, row-major, dtype bf16 or fp32;
 * counts: device, two 8-byte-aligned unsigned 64-bit counters the caller zeroes
 * and reads after a stream sync.  Argument errors as for cci_pack.
 */
cci_status cci_pack_stats(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K,
                          unsigned long long *counts, cci_stream_t stream);

/*
 * cci_linear_fused / cci_conv2d_fused -- the product / convolution of
 * cci_linear_ws / cci_conv2d_ws on a tensor-core family (the fused one where AUTO
 * would pick it or no workspace is given, else CCI_ALGO_DENSE_TC_WS), followed by the usual
 * output stage of a CNN layer, applied in the kernel's epilogue to each fp32
 * accumulator y[n][co] (the sum of Alg. 2, Sec. 3.2):
 *   y += bias[co]          when bias != NULL (fp32, Cout entries, 16-byte aligned);
 *   y = max(y, 0)          when relu != 0;
 *   Y[n][co] = y           as fp32 (out_dtype CCI_F32) or rounded to the nearest
 *                          bf16, ties to even (out_dtype CCI_BF16; needs Cout % 8 == 0).
 * The paper defines only the product; bias, ReLU and the bf16 output are the
 * surrounding network's, fused here so that a layer's output is written once at
 * the width the next layer reads.  X and Y must be 16-byte aligned and, for
 * layers without the fused family, the workspace as for CCI_ALGO_DENSE_TC_WS
 * (else CCI_ERR_ALIGN / CCI_ERR_WORKSPACE; the workspace may be NULL otherwise);
 * layers without that family return CCI_ERR_UNSUPPORTED.  Y is [N][Cout] or NHWC
 * [B][P][Q][Cout] of out_dtype; everything else as for cci_linear_ws /
 * cci_conv2d_ws.  NaN accumulators become 0 under the ReLU.
 */
cci_status cci_linear_fused(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                            const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                            const float *bias, int relu, cci_dtype out_dtype, void *Y,
                            uint32_t *dev_status, void *workspace, size_t workspace_bytes,
                            cci_stream_t stream);
cci_status cci_conv2d_fused(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W,
                            int64_t Cin, const void *values, const uint8_t *idx, int64_t Cout,
                            int KH, int KW, int stride_h, int stride_w, int pad_h, int pad_w,
                            int G, int K, const float *bias, int relu, cci_dtype out_dtype,
                            void *Y, uint32_t *dev_status, void *workspace,
                            size_t workspace_bytes, cci_stream_t stream);

/*
 * cci_dense_linear_tc / cci_dense_conv2d_tc -- the tensor-core GEMM of
 * CCI_ALGO_DENSE_TC_WS run on a DENSE weight matrix that the caller provides,
 * with no decompression: Y = X * Wd^T (a convolution: the implicit product of
 * cci_conv2d with Wd in OHWI order).  This is the reference line that isolates
 * what the sparsity buys on this hardware: Sec. 3.2 argues that CCI cuts the
 * work of the product by G/K; timing the same kernel on the unpruned weights
 * shows how much of that a dense tensor-core product keeps.
 *
 *   Wd   device, 16-byte aligned, in the workspace layout of the dense family
 *        (CCI_ALGO_DENSE_TC_WS): bf16 dense [Cout][R]; fp32 the two operand
 *        planes, as cci_dense_planes writes them
 *   X, Y as cci_linear / cci_conv2d, 16-byte aligned; Cin % 8 == 0 (bf16) or
 *        % 4 == 0 (fp32); Cout % 4 == 0
 * Errors: CCI_ERR_NULL, CCI_ERR_SHAPE, CCI_ERR_DTYPE, CCI_ERR_ALIGN,
 *         CCI_ERR_UNSUPPORTED (shapes the dense kernel lacks), CCI_ERR_CUDA.
 */
cci_status cci_dense_linear_tc(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *Wd,
                               int64_t Cout, float *Y, uint32_t *dev_status, cci_stream_t stream);
cci_status cci_dense_conv2d_tc(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W,
                               int64_t Cin, const void *Wd, int64_t Cout, int KH, int KW,
                               int stride_h, int stride_w, int pad_h, int pad_w, float *Y,
                               uint32_t *dev_status, cci_stream_t stream);

/*
 * cci_dense_planes -- writes a dense weight matrix W[Cout][R] (device, 16-byte
 * aligned, OHWI order for a convolution) in the workspace layout that
 * cci_dense_linear_tc / cci_dense_conv2d_tc read: bf16 copied as is; fp32 split
 * into the two operand planes of CCI_ALGO_DENSE_TC_WS (hi the nearest tf32 value
 * of w, lo = w - hi).  Wd: device, 16-byte aligned, bytes >=
 * cci_workspace_size(CCI_ALGO_DENSE_TC_WS, dtype, Cout, R).  Asynchronous on
 * stream.  Errors: CCI_ERR_DTYPE, CCI_ERR_SHAPE, CCI_ERR_NULL, CCI_ERR_WORKSPACE
 * (bytes too small), CCI_ERR_ALIGN (pointers, or R % 4 (fp32) / % 8 (bf16)),
 * CCI_ERR_CUDA.
 */
cci_status cci_dense_planes(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, void *Wd, size_t bytes,
                            cci_stream_t stream);

/* Largest dense-weight size (Cout*R*2 bytes) that cci_linear_dense_tc_static accepts. */
#define CCI_STATIC_WORKSPACE_BYTES (16u * 1024u * 1024u)

/*
 * cci_linear_dense_tc_static -- the product of cci_linear_ws with
 * CCI_ALGO_DENSE_TC_WS, for callers that cannot allocate device memory
 * themselves: for example a plug-in called by a host framework that owns all
 * device memory and hands it no allocator, or a latency-bound serving loop that
 * forbids allocations after start-up.  Such a caller still passes X, the packed
 * weights and Y, but no workspace: the dense weights are decompressed into a
 * scratch array that lives in the library itself (a static device array of
 * CCI_STATIC_WORKSPACE_BYTES, held by every GPU that loads the library until the
 * process exits).  This entry point calls no allocation routine.  (The paper
 * has no counterpart: this is a deployment convenience of this library.)
 *
 *   arguments  as cci_linear (bf16 only, Cin % 8 == 0, 16-byte aligned X and Y)
 * Rules:
 *   - Cout*Cin*2 > CCI_STATIC_WORKSPACE_BYTES is rejected with CCI_ERR_WORKSPACE;
 *   - the first call on a device looks up the array's device address on that
 *     device (the device current at the call); make that first call before any
 *     stream capture.  The address is cached for the life of the process: after
 *     cudaDeviceReset() on that device the cached address is stale, so do not
 *     call this entry point again on a device that was reset;
 *   - every call shares the one array per device and leaves it holding the last
 *     call's dense weights; each call rewrites the part it reads, so nothing
 *     needs clearing, but calls that overlap on the GPU (other streams, other
 *     threads) race on the array and must be serialised by the caller.
 * Errors: as cci_linear; CCI_ERR_UNSUPPORTED for shapes the dense kernel lacks;
 *         CCI_ERR_CUDA if the address lookup fails.
 */
cci_status cci_linear_dense_tc_static(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                                      const void *values, const uint8_t *idx, int64_t Cout, int G,
                                      int K, float *Y, uint32_t *dev_status, cci_stream_t stream);

/*
 * cci_kernel_name -- the name of the kernel family that cci_linear_ws /
 * cci_conv2d_ws would run for a layer with these sizes (R = Cin for a product,
 * Cin*KH*KW for a convolution, taken to have strides <= 2) when every pointer is
 * 16-byte aligned and, for CCI_ALGO_AUTO, the workspace is the one
 * cci_workspace_size(CCI_ALGO_AUTO) asks for: a static string, "" when the call
 * would be rejected.  No device work; used to label results.
 */
const char *cci_kernel_name(cci_dtype dtype, int64_t Cin, int64_t R, int64_t Cout, int G, int K,
                            cci_algo algo);

/* Human-readable text of a status code (static string). */
const char *cci_status_string(cci_status status);

/* The lowest-numbered error among the bits set in a device status word, or
 * CCI_OK when none is set. */
cci_status cci_decode_device_status(uint32_t word);

/* Library version, major*10000 + minor*100 + patch. */
int cci_version(void);

/*
 * cci_fma_probe -- measurement helper, not part of the method: enqueue one
 * kernel of `blocks` x `threads` threads, each running `iters` iterations of 16
 * independent packed fp32 FMAs (fma.rn.f32x2, 2 FMAs each), and write one float
 * per thread to `out` (device, blocks*threads floats) so the work is kept.
 * Flops performed = blocks * threads * iters * 64.  Time it with CUDA events to
 * measure the CUDA-core FMA throughput.
 * Errors: CCI_ERR_NULL, CCI_ERR_SHAPE, CCI_ERR_CUDA.
 */
cci_status cci_fma_probe(float *out, int blocks, int threads, int iters, cci_stream_t stream);

/*
 * cci_wait_probe -- diagnostic of the bounded waits inside the tensor-core
 * kernels (a safety mechanism of this library; the paper has no counterpart).
 * One thread initialises an mbarrier that expects one arrival, arrives on it if
 * `arrive` is nonzero, and waits for the barrier's phase exactly as the kernels
 * wait for their copies and MMAs.  With the arrival the wait returns at once and
 * nothing is reported.  Without it nothing can complete the phase: the wait
 * gives up after 2^31 SM clock cycles (about one second), ORs bit
 * (1u << CCI_ERR_TIMEOUT) into *dev_status and the kernel returns, leaving the
 * context usable.
 *   dev_status  device uint32, required
 * Errors: CCI_ERR_NULL, CCI_ERR_CUDA.
 */
cci_status cci_wait_probe(uint32_t *dev_status, int arrive, cci_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CCI_H_ */
