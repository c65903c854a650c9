// cci_api.cu -- the extern "C" entry points of libcci.so (declared in cci.h).
//
// Host side only: argument checks (all before anything is enqueued), choice of
// kernel, launch on the caller's stream.  The library allocates nothing.
#include <cstdint>
#include <cstring>
#include <mutex>

#include "cci_kernels.h"

namespace cci {

extern const RegtileEntry kRegtile_f32_a[];
extern const RegtileEntry kRegtile_f32_b[];
extern const RegtileEntry kRegtile_bf16_a[];
extern const RegtileEntry kRegtile_bf16_b[];

namespace {

constexpr int64_t kMaxElems = int64_t(1) << 62;

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

size_t elem_size(int dtype) { return dtype == CCI_F32 ? 4 : 2; }

bool valid_dtype(int dtype) { return dtype == CCI_F32 || dtype == CCI_BF16; }

// a*b without overflow past kMaxElems (all inputs >= 0)
bool mul_ok(int64_t a, int64_t b)
{
    if (a == 0 || b == 0) return true;
    return a <= kMaxElems / b;
}

cci_status check_group(int64_t Cout, int G, int K)
{
    if (G < 1 || G > 256 || K < 1 || K > G) return CCI_ERR_GROUP;
    if (Cout % G != 0) return CCI_ERR_GROUP;
    return CCI_OK;
}

// expand = true: the branch-free kernel (D == 0); false: the jump-dispatch kernel
const RegtileEntry *find_regtile(int dtype, int G, int K, bool expand)
{
    const RegtileEntry *tables[] = {kRegtile_f32_a, kRegtile_f32_b, kRegtile_bf16_a, kRegtile_bf16_b};
    for (const RegtileEntry *t : tables)
        for (; t->launch; ++t)
            if (t->dtype == dtype && t->G == G && t->K == K && (t->D == 0) == expand) return t;
    return nullptr;
}

// the register-tiled family AUTO uses (measured on GB300: the branch-free kernel
// is faster than the jump dispatch at every (G, K) of the workloads)
bool auto_prefers_expand(int dtype, int G, int K)
{
    (void)dtype;
    (void)G;
    (void)K;
    return true;
}

// shape conditions of the register-tiled kernel (16-byte vector copies)
bool regtile_shape_ok(int dtype, int64_t Cin, int64_t R, int K)
{
    const int64_t vec = 16 / static_cast<int64_t>(elem_size(dtype));
    return (Cin % vec == 0) && ((R * K) % 16 == 0) && (R < (int64_t(1) << 31));
}

bool regtile_ptr_ok(const FwdParams &p)
{
    return aligned(p.X, 16) && aligned(p.values, 16) && aligned(p.idx, 16) && aligned(p.Y, 16);
}

cci_status to_status(cudaError_t e) { return e == cudaSuccess ? CCI_OK : CCI_ERR_CUDA; }

// workspace of the dense tensor-core family: bf16 dense weights [Cout][R], or
// for fp32 the two operand planes of the split (cci_common.cuh): plane 0
// [Cout][R] of 4-byte elements, plane 1 [Cout][ceil(R / 32) * 64] of 2-byte ones
size_t dense_ws_bytes(int dtype, int64_t Cout, int64_t R)
{
    if (dtype == CCI_F32)
        return static_cast<size_t>(Cout) * (static_cast<size_t>(R) * 4 + static_cast<size_t>((R + 31) / 32) * 128);
    return static_cast<size_t>(Cout) * static_cast<size_t>(R) * 2;
}

bool dense_tc_shape_ok(int dtype, int G, int K, int64_t Cin, int64_t R)
{
    const int64_t v = dtype == CCI_F32 ? 4 : 8;  // elements per 16 bytes
    return dense_tc_supported(dtype, G, K) && Cin % v == 0 && R % v == 0;
}

// the dense tensor-core GEMM on caller weights p.wdense (no decompression)
cci_status dense_forward(FwdParams p, int dtype, cudaStream_t stream)
{
    if (p.is_conv && p.KH == 1 && p.KW == 1 && p.sh == 1 && p.sw == 1 && p.ph == 0 && p.pw == 0) p.is_conv = 0;
    const int64_t v = dtype == CCI_F32 ? 4 : 8;  // elements per 16 bytes
    if (p.R >= (int64_t(1) << 31) || p.Cout >= (int64_t(1) << 31) || p.Cin % v != 0 || p.R % v != 0 ||
        p.Cout % 4 != 0)
        return CCI_ERR_UNSUPPORTED;
    if (!aligned(p.X, 16) || !aligned(p.Y, 16) || !aligned(p.wdense, 16)) return CCI_ERR_ALIGN;
    if (p.N == 0) return CCI_OK;
    return to_status(launch_gemm_ws(p, dtype, stream));
}

// the fused tensor-core family (packed weights expanded in the GEMM, no
// workspace) may have this layer: bf16, a dense-kernel shape, 16-byte aligned
// operands and the expansion's conditions (gemm_pk_shape_ok); whether its
// activations can be copied by TMA is settled by launch_gemm_pk, which returns
// cudaErrorNotSupported before launching anything when they cannot
bool fused_may(const FwdParams &p, int dtype)
{
    const bool tc_fits = p.R < (int64_t(1) << 31) && p.Cout < (int64_t(1) << 31);
    return dtype == CCI_BF16 && tc_fits && p.Cin % 8 == 0 && p.R % 8 == 0 && p.Cout % 4 == 0 && aligned(p.X, 16) &&
           aligned(p.Y, 16) && gemm_pk_shape_ok(p);
}

// the entry points with an output epilogue (cci_linear_fused, cci_conv2d_fused):
// a tensor-core family, whatever the epilogue flags
constexpr cci_algo kAlgoEpilogue = static_cast<cci_algo>(100);

// AUTO takes the fused family over the workspace family when the caller gives a
// workspace only where it measured faster on GB300: nowhere yet (the K/G sweep
// point G = 8, K = 2: 0.57 ms fused against 0.16 ms decompression + GEMM), so
// with a workspace AUTO runs the workspace family, without one the fused family
bool auto_prefers_fused(int K)
{
    (void)K;
    return false;
}

// 1: the fused kernel was launched, 0: the layer does not have it (nothing
// enqueued), -1: launch error
int try_fused(const FwdParams &p, int dtype, cudaStream_t stream)
{
    if (!fused_may(p, dtype)) return 0;
    const cudaError_t e = launch_gemm_pk(p, stream);
    if (e == cudaErrorNotSupported) return 0;
    return e == cudaSuccess ? 1 : -1;
}

cci_status fused_status(int r) { return r > 0 ? CCI_OK : CCI_ERR_CUDA; }

cci_status forward(FwdParams p, int dtype, int G, int K, cci_algo algo, void *ws, size_t ws_bytes,
                   cudaStream_t stream)
{
    // a 1x1 convolution with unit stride and no padding is the product of X[B*H*W][Cin]
    if (p.is_conv && p.KH == 1 && p.KW == 1 && p.sh == 1 && p.sw == 1 && p.ph == 0 && p.pw == 0) p.is_conv = 0;
    p.G = G;
    p.K = K;
    const bool tc_fits = p.R < (int64_t(1) << 31) && p.Cout < (int64_t(1) << 31);  // 32-bit copy coordinates
    const bool ws_ok = ws && ws_bytes >= dense_ws_bytes(dtype, p.Cout, p.R) && aligned(ws, 16);
    const bool dense_ok = tc_fits && dense_tc_shape_ok(dtype, G, K, p.Cin, p.R);
    if (algo == kAlgoEpilogue || p.bias || p.relu || p.out_bf16) {
        // the output epilogue exists on the tensor-core families: the fused one when
        // the layer has it (preferred as for AUTO, or when no workspace is given),
        // else the workspace one
        if (!dense_ok) return CCI_ERR_UNSUPPORTED;
        if (p.out_bf16 && p.Cout % 8 != 0) return CCI_ERR_UNSUPPORTED;  // 16-byte output rows
        if (p.bias && !aligned(p.bias, 16)) return CCI_ERR_ALIGN;
        if (!aligned(p.X, 16) || !aligned(p.Y, 16)) return CCI_ERR_ALIGN;
        if (p.N == 0) return CCI_OK;
        if (auto_prefers_fused(K) || !ws_ok) {
            const int r = try_fused(p, dtype, stream);
            if (r != 0) return fused_status(r);
        }
        if (!ws_ok) return CCI_ERR_WORKSPACE;
        algo = CCI_ALGO_DENSE_TC_WS;
    }
    if (p.N == 0) return CCI_OK;
    if (algo == CCI_ALGO_AUTO) {
        if (auto_prefers_fused(K)) {
            const int r = try_fused(p, dtype, stream);
            if (r != 0) return fused_status(r);
        }
        if (dense_ok && ws_ok && aligned(p.X, 16) && aligned(p.Y, 16)) {
            algo = CCI_ALGO_DENSE_TC_WS;
        } else if (!auto_prefers_fused(K)) {
            const int r = try_fused(p, dtype, stream);
            if (r != 0) return fused_status(r);
        }
    }
    if (algo == CCI_ALGO_DENSE_TC) {
        const int r = try_fused(p, dtype, stream);
        return r == 0 ? CCI_ERR_UNSUPPORTED : fused_status(r);
    }
    if (algo == CCI_ALGO_DENSE_TC_WS) {
        if (!tc_fits || !dense_tc_shape_ok(dtype, G, K, p.Cin, p.R) || !aligned(p.X, 16) || !aligned(p.Y, 16))
            return CCI_ERR_UNSUPPORTED;
        if (!ws_ok) return CCI_ERR_WORKSPACE;
        p.wdense = ws;
        return to_status(launch_dense_tc_ws(p, dtype, G, K, stream));
    }
    if (algo == CCI_ALGO_AUTO || algo == CCI_ALGO_REGTILE || algo == CCI_ALGO_EXPAND) {
        const bool expand = algo == CCI_ALGO_EXPAND || (algo == CCI_ALGO_AUTO && auto_prefers_expand(dtype, G, K));
        const RegtileEntry *e = find_regtile(dtype, G, K, expand);
        if (e && regtile_shape_ok(dtype, p.Cin, p.R, K) && regtile_ptr_ok(p)) return to_status(e->launch(p, stream));
        if (algo != CCI_ALGO_AUTO) return CCI_ERR_UNSUPPORTED;
    } else if (algo != CCI_ALGO_GENERIC) {
        return CCI_ERR_UNSUPPORTED;
    }
    return to_status(launch_generic(p, dtype, G, K, stream));
}

cci_status check_common(const void *X, int dtype, const void *values, const uint8_t *idx, float *Y,
                        int64_t N, int64_t Cout, int64_t R, int G, int K)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!values || !idx) return CCI_ERR_NULL;
    if (N > 0 && (!X || !Y)) return CCI_ERR_NULL;
    if (N < 0 || Cout < 1 || R < 1) return CCI_ERR_SHAPE;
    const cci_status g = check_group(Cout, G, K);
    if (g != CCI_OK) return g;
    if (!mul_ok(N, Cout) || !mul_ok(R, K) || !mul_ok(R * K, Cout / G) || R >= (int64_t(1) << 40))
        return CCI_ERR_SHAPE;
    const size_t es = elem_size(dtype);
    if (!aligned(values, es) || (X && !aligned(X, es)) || (Y && !aligned(Y, 4))) return CCI_ERR_ALIGN;
    return CCI_OK;
}

}  // namespace

int regtile_wc(int64_t groups, int MG)
{
    // 8 channel-warps when the layer has enough groups, else 4 (fewer would
    // widen the column tile past the shared-memory budget)
    return static_cast<int64_t>(8) * MG <= groups ? 8 : 4;
}

}  // namespace cci

using namespace cci;

extern "C" {

int cci_version(void) { return 1 * 10000 + 0 * 100 + 0; }

const char *cci_status_string(cci_status s)
{
    switch (s) {
        case CCI_OK: return "ok";
        case CCI_ERR_NULL: return "a required pointer is NULL";
        case CCI_ERR_SHAPE: return "invalid or too large shape";
        case CCI_ERR_GROUP: return "invalid group: need 1 <= K <= G <= 256 and Cout % G == 0";
        case CCI_ERR_DTYPE: return "unknown dtype";
        case CCI_ERR_ALIGN: return "pointer not aligned to its element size";
        case CCI_ERR_VALUE: return "NaN among the weights given to cci_pack";
        case CCI_ERR_CUDA: return "CUDA launch or runtime error";
        case CCI_ERR_TIMEOUT: return "a bounded wait inside a kernel expired";
        case CCI_ERR_UNSUPPORTED: return "request not supported by this build";
        case CCI_ERR_INDEX: return "a packed index >= G (dense kernels: or not strictly increasing)";
        case CCI_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    }
    return "unknown status";
}

cci_status cci_decode_device_status(uint32_t word)
{
    for (int b = 1; b < 32; ++b)
        if (word & (1u << b)) return static_cast<cci_status>(b);
    return CCI_OK;
}

cci_status cci_pack(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                    uint8_t *idx, uint32_t *dev_status, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!W || !values || !idx) return CCI_ERR_NULL;
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return CCI_ERR_SHAPE;
    const cci_status g = check_group(Cout, G, K);
    if (g != CCI_OK) return g;
    const size_t es = elem_size(dtype);
    if (!aligned(W, es) || !aligned(values, es)) return CCI_ERR_ALIGN;
    return to_status(launch_pack(W, dtype, Cout, R, G, K, values, idx, dev_status,
                                 reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"

namespace {

struct Epilogue {
    const float *bias;
    int relu;
    int out_bf16;
};

// parameters of the product Y[N][Cout] = X[N][Cin] * Wd^T (fp32 output, no epilogue)
FwdParams linear_params(const void *X, int64_t N, int64_t Cin, const void *values, const uint8_t *idx,
                        int64_t Cout, float *Y, uint32_t *dev_status)
{
    FwdParams p{};
    p.X = X;
    p.values = values;
    p.idx = idx;
    p.Y = Y;
    p.status = dev_status;
    p.N = N;
    p.Cout = Cout;
    p.R = Cin;
    p.Cin = Cin;
    p.H = p.W = p.P = p.Q = 1;
    p.KH = p.KW = p.sh = p.sw = 1;
    p.ph = p.pw = 0;
    p.is_conv = 0;
    return p;
}

cci_status linear_impl(const void *X, int dtype, int64_t N, int64_t Cin, const void *values, const uint8_t *idx,
                       int64_t Cout, int G, int K, void *Y, uint32_t *dev_status, cci_algo algo, void *workspace,
                       size_t workspace_bytes, cci_stream_t stream, Epilogue e)
{
    const cci_status st = check_common(X, dtype, values, idx, static_cast<float *>(Y), N, Cout, Cin, G, K);
    if (st != CCI_OK) return st;
    if (!mul_ok(N, Cin)) return CCI_ERR_SHAPE;
    FwdParams p = linear_params(X, N, Cin, values, idx, Cout, static_cast<float *>(Y), dev_status);
    p.bias = e.bias;
    p.relu = e.relu;
    p.out_bf16 = e.out_bf16;
    return forward(p, dtype, G, K, algo, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

cci_status conv_impl(const void *X, int dtype, int64_t B, int64_t H, int64_t W, int64_t Cin, const void *values,
                     const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h, int stride_w, int pad_h,
                     int pad_w, int G, int K, void *Y, uint32_t *dev_status, cci_algo algo, void *workspace,
                     size_t workspace_bytes, cci_stream_t stream, Epilogue e);

// geometry of a convolution (cross-correlation, zero padding, floor output size)
// into p: sizes, strides, padding, N = B*P*Q and R = KH*KW*Cin; CCI_ERR_SHAPE for
// sizes out of range or without an output
cci_status conv_params(int64_t B, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int KH, int KW, int stride_h,
                       int stride_w, int pad_h, int pad_w, FwdParams *p)
{
    if (B < 0 || H < 1 || W < 1 || Cin < 1 || Cout < 1 || KH < 1 || KW < 1 || stride_h < 1 || stride_w < 1 ||
        pad_h < 0 || pad_w < 0)
        return CCI_ERR_SHAPE;
    const int64_t lim = int64_t(1) << 30;
    if (H >= lim || W >= lim || pad_h >= lim || pad_w >= lim) return CCI_ERR_SHAPE;
    if (H + 2 * pad_h < KH || W + 2 * pad_w < KW) return CCI_ERR_SHAPE;
    const int64_t P = (H + 2 * pad_h - KH) / stride_h + 1;
    const int64_t Q = (W + 2 * pad_w - KW) / stride_w + 1;
    if (!mul_ok(P, Q) || !mul_ok(B, P * Q) || !mul_ok(H, W) || !mul_ok(H * W, Cin) || !mul_ok(B, H * W * Cin) ||
        !mul_ok(static_cast<int64_t>(KH) * KW, Cin))
        return CCI_ERR_SHAPE;
    p->N = B * P * Q;
    p->Cout = Cout;
    p->R = static_cast<int64_t>(KH) * KW * Cin;
    p->Cin = Cin;
    p->H = H;
    p->W = W;
    p->P = P;
    p->Q = Q;
    p->KH = KH;
    p->KW = KW;
    p->sh = stride_h;
    p->sw = stride_w;
    p->ph = pad_h;
    p->pw = pad_w;
    p->is_conv = 1;
    return CCI_OK;
}

}  // namespace

extern "C" {

cci_status cci_td_mask(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K, float rate,
                       const float *uniforms, void *W_out, uint8_t *mask, uint32_t *dev_status, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!W || !uniforms || !W_out) return CCI_ERR_NULL;
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return CCI_ERR_SHAPE;
    const cci_status g = check_group(Cout, G, K);
    if (g != CCI_OK) return g;
    if (!(rate >= 0.0f && rate <= 1.0f)) return CCI_ERR_VALUE;  // also NaN
    const size_t es = elem_size(dtype);
    if (!aligned(W, es) || !aligned(W_out, es) || !aligned(uniforms, 4)) return CCI_ERR_ALIGN;
    return to_status(launch_td_mask(W, dtype, Cout, R, G, K, rate, uniforms, W_out, mask, dev_status,
                                    reinterpret_cast<cudaStream_t>(stream)));
}

float cci_td_drop_rate(int64_t step, int64_t ramp_steps, float start, float end)
{
    if (ramp_steps <= 0) return end;
    const int64_t s = step < 0 ? 0 : (step > ramp_steps ? ramp_steps : step);
    return start + (end - start) * static_cast<float>(static_cast<double>(s) / static_cast<double>(ramp_steps));
}

cci_status cci_bbs_pack(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                        uint8_t *idx, uint32_t *dev_status, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!W || !values || !idx) return CCI_ERR_NULL;
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return CCI_ERR_SHAPE;
    if (G < 1 || G > 256 || K < 1 || K > G || R % G != 0) return CCI_ERR_GROUP;
    const size_t es = elem_size(dtype);
    if (!aligned(W, es) || !aligned(values, es)) return CCI_ERR_ALIGN;
    return to_status(launch_bbs_pack(W, dtype, Cout, R, G, K, values, idx, dev_status,
                                     reinterpret_cast<cudaStream_t>(stream)));
}

cci_status cci_bbs_linear(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                          const uint8_t *idx, int64_t Cout, int G, int K, float *Y, uint32_t *dev_status,
                          cci_algo algo, void *workspace, size_t workspace_bytes, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!values || !idx) return CCI_ERR_NULL;
    if (N > 0 && (!X || !Y)) return CCI_ERR_NULL;
    if (N < 0 || Cout < 1 || Cin < 1 || !mul_ok(N, Cout) || !mul_ok(N, Cin) || !mul_ok(Cout, Cin))
        return CCI_ERR_SHAPE;
    if (G < 1 || G > 256 || K < 1 || K > G || Cin % G != 0) return CCI_ERR_GROUP;
    const size_t es = elem_size(dtype);
    if (!aligned(values, es) || (X && !aligned(X, es)) || (Y && !aligned(Y, 4))) return CCI_ERR_ALIGN;
    FwdParams p{};
    p.X = X;
    p.values = values;
    p.idx = idx;
    p.Y = Y;
    p.status = dev_status;
    p.N = N;
    p.Cout = Cout;
    p.R = Cin;
    p.Cin = Cin;
    p.H = p.W = p.P = p.Q = 1;
    p.KH = p.KW = p.sh = p.sw = 1;
    const int64_t v = dtype == CCI_F32 ? 4 : 8;  // elements per 16 bytes
    const bool tc_ok = Cin % v == 0 && Cin < (int64_t(1) << 31) && Cout < (int64_t(1) << 31) &&
                       Cout % 4 == 0 && aligned(X, 16) && aligned(Y, 16);
    const bool ws_ok = workspace && workspace_bytes >= dense_ws_bytes(dtype, Cout, Cin) && aligned(workspace, 16);
    if (algo == CCI_ALGO_AUTO) algo = (tc_ok && ws_ok) ? CCI_ALGO_DENSE_TC_WS : CCI_ALGO_GENERIC;
    if (algo == CCI_ALGO_DENSE_TC_WS) {
        if (!tc_ok) return CCI_ERR_UNSUPPORTED;
        if (!ws_ok) return CCI_ERR_WORKSPACE;
        if (N == 0) return CCI_OK;
        p.wdense = workspace;
        const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
        const cudaError_t e = launch_bbs_decompress(p, dtype, G, K, s);
        if (e != cudaSuccess) return CCI_ERR_CUDA;
        return to_status(launch_gemm_ws(p, dtype, s));
    }
    if (algo != CCI_ALGO_GENERIC || 32 % G != 0) return CCI_ERR_UNSUPPORTED;
    if (N == 0) return CCI_OK;
    return to_status(launch_bbs_gather(p, dtype, G, K, reinterpret_cast<cudaStream_t>(stream)));
}

cci_status cci_pack_stats(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, int G, int K,
                          unsigned long long *counts, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!W || !counts) return CCI_ERR_NULL;
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return CCI_ERR_SHAPE;
    const cci_status g = check_group(Cout, G, K);
    if (g != CCI_OK) return g;
    if (!aligned(W, elem_size(dtype)) || !aligned(counts, 8)) return CCI_ERR_ALIGN;
    return to_status(launch_pack_stats(W, dtype, Cout, R, G, K, counts, reinterpret_cast<cudaStream_t>(stream)));
}

cci_status cci_linear_ws(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                         const uint8_t *idx, int64_t Cout, int G, int K, float *Y, uint32_t *dev_status,
                         cci_algo algo, void *workspace, size_t workspace_bytes, cci_stream_t stream)
{
    return linear_impl(X, dtype, N, Cin, values, idx, Cout, G, K, Y, dev_status, algo, workspace, workspace_bytes,
                       stream, Epilogue{nullptr, 0, 0});
}

cci_status cci_linear_fused(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                            const uint8_t *idx, int64_t Cout, int G, int K, const float *bias, int relu,
                            cci_dtype out_dtype, void *Y, uint32_t *dev_status, void *workspace,
                            size_t workspace_bytes, cci_stream_t stream)
{
    if (!valid_dtype(out_dtype)) return CCI_ERR_DTYPE;
    return linear_impl(X, dtype, N, Cin, values, idx, Cout, G, K, Y, dev_status, kAlgoEpilogue, workspace,
                       workspace_bytes, stream, Epilogue{bias, relu != 0, out_dtype == CCI_BF16});
}

cci_status cci_linear_ex(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                         const uint8_t *idx, int64_t Cout, int G, int K, float *Y, uint32_t *dev_status,
                         cci_algo algo, cci_stream_t stream)
{
    return cci_linear_ws(X, dtype, N, Cin, values, idx, Cout, G, K, Y, dev_status, algo, nullptr, 0, stream);
}

cci_status cci_linear(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *values,
                      const uint8_t *idx, int64_t Cout, int G, int K, float *Y, uint32_t *dev_status,
                      cci_stream_t stream)
{
    return cci_linear_ex(X, dtype, N, Cin, values, idx, Cout, G, K, Y, dev_status, CCI_ALGO_AUTO, stream);
}

cci_status cci_conv2d_ws(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W, int64_t Cin,
                         const void *values, const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h,
                         int stride_w, int pad_h, int pad_w, int G, int K, float *Y, uint32_t *dev_status,
                         cci_algo algo, void *workspace, size_t workspace_bytes, cci_stream_t stream)
{
    return conv_impl(X, dtype, B, H, W, Cin, values, idx, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, G, K, Y,
                     dev_status, algo, workspace, workspace_bytes, stream, Epilogue{nullptr, 0, 0});
}

cci_status cci_conv2d_fused(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W, int64_t Cin,
                            const void *values, const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h,
                            int stride_w, int pad_h, int pad_w, int G, int K, const float *bias, int relu,
                            cci_dtype out_dtype, void *Y, uint32_t *dev_status, void *workspace,
                            size_t workspace_bytes, cci_stream_t stream)
{
    if (!valid_dtype(out_dtype)) return CCI_ERR_DTYPE;
    return conv_impl(X, dtype, B, H, W, Cin, values, idx, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, G, K, Y,
                     dev_status, kAlgoEpilogue, workspace, workspace_bytes, stream,
                     Epilogue{bias, relu != 0, out_dtype == CCI_BF16});
}

}  // extern "C"

namespace {

cci_status conv_impl(const void *X, int dtype, int64_t B, int64_t H, int64_t W, int64_t Cin, const void *values,
                     const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h, int stride_w, int pad_h,
                     int pad_w, int G, int K, void *Y_, uint32_t *dev_status, cci_algo algo, void *workspace,
                     size_t workspace_bytes, cci_stream_t stream, Epilogue e)
{
    float *Y = static_cast<float *>(Y_);
    FwdParams p{};
    const cci_status geo = conv_params(B, H, W, Cin, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, &p);
    if (geo != CCI_OK) return valid_dtype(dtype) ? geo : CCI_ERR_DTYPE;
    const cci_status st = check_common(X, dtype, values, idx, Y, p.N, Cout, p.R, G, K);
    if (st != CCI_OK) return st;
    p.X = X;
    p.values = values;
    p.idx = idx;
    p.Y = Y;
    p.status = dev_status;
    p.bias = e.bias;
    p.relu = e.relu;
    p.out_bf16 = e.out_bf16;
    return forward(p, dtype, G, K, algo, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
}

}  // namespace

extern "C" {

cci_status cci_conv2d_ex(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W, int64_t Cin,
                         const void *values, const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h,
                         int stride_w, int pad_h, int pad_w, int G, int K, float *Y, uint32_t *dev_status,
                         cci_algo algo, cci_stream_t stream)
{
    return cci_conv2d_ws(X, dtype, B, H, W, Cin, values, idx, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, G, K,
                         Y, dev_status, algo, nullptr, 0, stream);
}

size_t cci_workspace_size(cci_algo algo, cci_dtype dtype, int64_t Cout, int64_t R)
{
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return 0;
    if (!valid_dtype(dtype)) return 0;
    if (algo == CCI_ALGO_DENSE_TC_WS || algo == CCI_ALGO_AUTO) return dense_ws_bytes(dtype, Cout, R);
    return 0;
}

cci_status cci_conv2d(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W, int64_t Cin,
                      const void *values, const uint8_t *idx, int64_t Cout, int KH, int KW, int stride_h,
                      int stride_w, int pad_h, int pad_w, int G, int K, float *Y, uint32_t *dev_status,
                      cci_stream_t stream)
{
    return cci_conv2d_ex(X, dtype, B, H, W, Cin, values, idx, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, G, K,
                         Y, dev_status, CCI_ALGO_AUTO, stream);
}

cci_status cci_dense_linear_tc(const void *X, cci_dtype dtype, int64_t N, int64_t Cin, const void *Wd,
                               int64_t Cout, float *Y, uint32_t *dev_status, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!Wd || (N > 0 && (!X || !Y))) return CCI_ERR_NULL;
    if (N < 0 || Cin < 1 || Cout < 1 || !mul_ok(N, Cin) || !mul_ok(N, Cout) || !mul_ok(Cout, Cin))
        return CCI_ERR_SHAPE;
    FwdParams p = linear_params(X, N, Cin, nullptr, nullptr, Cout, Y, dev_status);
    p.wdense = Wd;
    return dense_forward(p, dtype, reinterpret_cast<cudaStream_t>(stream));
}

cci_status cci_dense_planes(const void *W, cci_dtype dtype, int64_t Cout, int64_t R, void *Wd, size_t bytes,
                            cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (Cout < 1 || R < 1 || !mul_ok(Cout, R)) return CCI_ERR_SHAPE;
    if (!W || !Wd) return CCI_ERR_NULL;
    if (bytes < dense_ws_bytes(dtype, Cout, R)) return CCI_ERR_WORKSPACE;
    if (!aligned(W, 16) || !aligned(Wd, 16) || R % (dtype == CCI_F32 ? 4 : 8) != 0) return CCI_ERR_ALIGN;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (dtype == CCI_BF16)
        return to_status(cudaMemcpyAsync(Wd, W, static_cast<size_t>(Cout) * R * 2, cudaMemcpyDeviceToDevice, st));
    return to_status(launch_dense_split(static_cast<const uint32_t *>(W), Cout, R, Wd, st));
}

cci_status cci_dense_conv2d_tc(const void *X, cci_dtype dtype, int64_t B, int64_t H, int64_t W, int64_t Cin,
                               const void *Wd, int64_t Cout, int KH, int KW, int stride_h, int stride_w, int pad_h,
                               int pad_w, float *Y, uint32_t *dev_status, cci_stream_t stream)
{
    if (!valid_dtype(dtype)) return CCI_ERR_DTYPE;
    if (!Wd || (B > 0 && (!X || !Y))) return CCI_ERR_NULL;
    FwdParams p{};
    const cci_status st = conv_params(B, H, W, Cin, Cout, KH, KW, stride_h, stride_w, pad_h, pad_w, &p);
    if (st != CCI_OK) return st;
    if (!mul_ok(Cout, p.R)) return CCI_ERR_SHAPE;
    p.X = X;
    p.Y = Y;
    p.status = dev_status;
    p.wdense = Wd;
    return dense_forward(p, dtype, reinterpret_cast<cudaStream_t>(stream));
}

namespace {

// name of the fused tensor-core kernel for a layer, "" when it has none
// (convolutions: as if the strides were at most 2, the condition of its
// activation copies)
const char *fused_name(int dtype, int64_t Cin, int64_t R, int64_t Cout, int G, int K)
{
    static const char *names[] = {"dense_tc_fused_bf16_G4_K1",  "dense_tc_fused_bf16_G4_K2",
                                  "dense_tc_fused_bf16_G8_K1",  "dense_tc_fused_bf16_G8_K2",
                                  "dense_tc_fused_bf16_G8_K4",  "dense_tc_fused_bf16_G16_K1",
                                  "dense_tc_fused_bf16_G16_K2", "dense_tc_fused_bf16_G16_K4",
                                  "dense_tc_fused_bf16_G16_K8", "dense_tc_fused_bf16_G32_K1",
                                  "dense_tc_fused_bf16_G32_K2", "dense_tc_fused_bf16_G32_K4",
                                  "dense_tc_fused_bf16_G32_K8"};
    if (dtype != CCI_BF16 || Cin % 8 != 0 || R % 8 != 0 || Cout % 4 != 0 || Cout % G != 0) return "";
    if (R >= (int64_t(1) << 31) || Cout >= (int64_t(1) << 31)) return "";
    FwdParams p{};
    p.values = reinterpret_cast<const void *>(uintptr_t(256));
    p.idx = reinterpret_cast<const uint8_t *>(uintptr_t(256));
    p.R = R;
    p.G = G;
    p.K = K;
    if (!gemm_pk_shape_ok(p)) return "";
    // activations copied by TMA: any product; a convolution (other than 1x1 with
    // unit stride, which is a product) when Cin is a multiple of the 64-deep stage
    if (R != Cin && Cin % 64 != 0) return "";
    int i = 0;
    for (int g = 4; g <= 32; g *= 2)
        for (int k = 1; k <= g / 2 && k <= 8; k *= 2, ++i)
            if (g == G && k == K) return names[i];
    return "";
}

}  // namespace

const char *cci_kernel_name(cci_dtype dtype, int64_t Cin, int64_t R, int64_t Cout, int G, int K, cci_algo algo)
{
    if (!valid_dtype(dtype) || Cin < 1 || R < Cin || check_group(Cout, G, K) != CCI_OK) return "";
    if (algo == CCI_ALGO_DENSE_TC_WS) {
        static const char *names_ws[] = {"dense_tc_ws_bf16_G4_K1", "dense_tc_ws_bf16_G4_K2", "dense_tc_ws_bf16_G8_K1",
                                         "dense_tc_ws_bf16_G8_K2", "dense_tc_ws_bf16_G8_K4", "dense_tc_ws_bf16_G16_K1",
                                         "dense_tc_ws_bf16_G16_K2", "dense_tc_ws_bf16_G16_K4", "dense_tc_ws_bf16_G16_K8",
                                         "dense_tc_ws_bf16_G32_K1", "dense_tc_ws_bf16_G32_K2", "dense_tc_ws_bf16_G32_K4",
                                         "dense_tc_ws_bf16_G32_K8", "dense_tc_ws_bf16_G32_K16"};
        static const char *names_tf[] = {"dense_tc_ws_f32split_G4_K1", "dense_tc_ws_f32split_G4_K2",
                                         "dense_tc_ws_f32split_G8_K1", "dense_tc_ws_f32split_G8_K2",
                                         "dense_tc_ws_f32split_G8_K4", "dense_tc_ws_f32split_G16_K1",
                                         "dense_tc_ws_f32split_G16_K2", "dense_tc_ws_f32split_G16_K4",
                                         "dense_tc_ws_f32split_G16_K8", "dense_tc_ws_f32split_G32_K1",
                                         "dense_tc_ws_f32split_G32_K2", "dense_tc_ws_f32split_G32_K4",
                                         "dense_tc_ws_f32split_G32_K8", "dense_tc_ws_f32split_G32_K16"};
        if (!dense_tc_shape_ok(dtype, G, K, Cin, R)) return "";
        int i = 0;
        for (int g = 4; g <= 32; g *= 2)
            for (int k = 1; k <= g / 2; k *= 2, ++i)
                if (g == G && k == K) return dtype == CCI_F32 ? names_tf[i] : names_ws[i];
        return "";
    }
    const char *fused = fused_name(dtype, Cin, R, Cout, G, K);
    if (algo == CCI_ALGO_DENSE_TC) return fused;
    if (algo == CCI_ALGO_AUTO) {
        // the family AUTO runs when given the workspace cci_workspace_size asks for
        if (fused[0] && auto_prefers_fused(K)) return fused;
        const char *ws = cci_kernel_name(dtype, Cin, R, Cout, G, K, CCI_ALGO_DENSE_TC_WS);
        if (ws[0]) return ws;
        if (fused[0]) return fused;
    }
    if (algo == CCI_ALGO_AUTO || algo == CCI_ALGO_REGTILE || algo == CCI_ALGO_EXPAND) {
        const bool expand = algo == CCI_ALGO_EXPAND || (algo == CCI_ALGO_AUTO && auto_prefers_expand(dtype, G, K));
        const RegtileEntry *e = find_regtile(dtype, G, K, expand);
        if (e && regtile_shape_ok(dtype, Cin, R, K)) return e->name;
        if (algo != CCI_ALGO_AUTO) return "";
    } else if (algo != CCI_ALGO_GENERIC) {
        return "";
    }
    return dtype == CCI_F32 ? "generic_f32" : "generic_bf16";
}

cci_status cci_fma_probe(float *out, int blocks, int threads, int iters, cci_stream_t stream)
{
    if (!out) return CCI_ERR_NULL;
    if (blocks < 1 || threads < 1 || threads > 1024 || iters < 0) return CCI_ERR_SHAPE;
    return to_status(launch_fma_probe(out, blocks, threads, iters, reinterpret_cast<cudaStream_t>(stream)));
}

cci_status cci_wait_probe(uint32_t *dev_status, int arrive, cci_stream_t stream)
{
    if (!dev_status) return CCI_ERR_NULL;
    return to_status(launch_wait_probe(dev_status, arrive, reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Static-scratch product for callers that cannot allocate device memory.
// The dense-weight scratch is this file-scope device array; host code here
// looks up its device address once per device (cudaGetSymbolAddress, with that
// device current) and passes the address to the kernels as their workspace.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kStaticWsBytes = CCI_STATIC_WORKSPACE_BYTES;
static __device__ __align__(256) unsigned char g_static_ws[kStaticWsBytes];

constexpr int kMaxDevices = 64;
std::mutex g_static_ws_mutex;
void *g_static_ws_ptr[kMaxDevices] = {};

// device address of g_static_ws on the current device (looked up on first use)
cci_status static_ws_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return CCI_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_static_ws_mutex);
    if (!g_static_ws_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_ws) != cudaSuccess || !p) return CCI_ERR_CUDA;
        g_static_ws_ptr[dev] = p;
    }
    *out = g_static_ws_ptr[dev];
    return CCI_OK;
}

}  // namespace

extern "C" cci_status cci_linear_dense_tc_static(const void *X, cci_dtype dtype, int64_t N, int64_t Cin,
                                                 const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                                                 float *Y, uint32_t *dev_status, cci_stream_t stream)
{
    const cci_status st = check_common(X, dtype, values, idx, Y, N, Cout, Cin, G, K);
    if (st != CCI_OK) return st;
    if (dtype != CCI_BF16) return CCI_ERR_UNSUPPORTED;  // the array holds bf16 dense weights
    if (!mul_ok(N, Cin) || !mul_ok(Cout, Cin)) return CCI_ERR_SHAPE;
    // shapes outside the dense kernel's limits are unsupported whatever their size;
    // only then is the size compared with the array (Cout * Cin cannot wrap here)
    if (Cin >= (int64_t(1) << 31) || Cout >= (int64_t(1) << 31) || !dense_tc_shape_ok(dtype, G, K, Cin, Cin))
        return CCI_ERR_UNSUPPORTED;
    if (dense_ws_bytes(dtype, Cout, Cin) > kStaticWsBytes) return CCI_ERR_WORKSPACE;
    if (N == 0) return CCI_OK;
    void *ws = nullptr;
    const cci_status a = static_ws_address(&ws);
    if (a != CCI_OK) return a;
    return cci_linear_ws(X, dtype, N, Cin, values, idx, Cout, G, K, Y, dev_status, CCI_ALGO_DENSE_TC_WS, ws,
                         kStaticWsBytes, stream);
}

// ---------------------------------------------------------------------------
// The product over host buffers: X read from host memory and Y written back to
// it, in chunks of columns pipelined over three streams (copy in, product, copy
// out) so that the copies of one chunk overlap the product of another.  The
// caller's device buffer holds the dense-weight workspace and two staging slots
// per direction.
// ---------------------------------------------------------------------------
namespace {

constexpr int kHostSlots = 2;  // staging slots per direction: chunk c + 1 in, c computed, c - 1 out

size_t round256(size_t b) { return (b + 255) / 256 * 256; }

struct HostLayout {
    size_t ws, xslot, yslot, total;
};

bool host_layout(int dtype, int64_t Cin, int64_t Cout, int64_t chunk, HostLayout *l)
{
    if (!valid_dtype(dtype) || Cin < 1 || Cout < 1 || chunk < 1 || !mul_ok(chunk, Cin) || !mul_ok(chunk, Cout) ||
        !mul_ok(Cout, Cin))
        return false;
    l->ws = round256(dense_ws_bytes(dtype, Cout, Cin));
    l->xslot = round256(static_cast<size_t>(chunk) * static_cast<size_t>(Cin) * elem_size(dtype));
    l->yslot = round256(static_cast<size_t>(chunk) * static_cast<size_t>(Cout) * 4);
    l->total = l->ws + kHostSlots * (l->xslot + l->yslot);
    return true;
}

}  // namespace

extern "C" size_t cci_linear_host_buffer_size(cci_dtype dtype, int64_t Cin, int64_t Cout, int64_t chunk_cols)
{
    HostLayout l;
    return host_layout(dtype, Cin, Cout, chunk_cols, &l) ? l.total : 0;
}

extern "C" cci_status cci_linear_host(const void *X_host, cci_dtype dtype, int64_t N, int64_t Cin,
                                      const void *values, const uint8_t *idx, int64_t Cout, int G, int K,
                                      float *Y_host, int64_t chunk_cols, void *device_buffer,
                                      size_t device_buffer_bytes, uint32_t *dev_status, cci_stream_t stream,
                                      cci_stream_t copy_in_stream, cci_stream_t copy_out_stream)
{
    const cci_status st = check_common(X_host, dtype, values, idx, Y_host, N, Cout, Cin, G, K);
    if (st != CCI_OK) return st;
    if (!mul_ok(N, Cin)) return CCI_ERR_SHAPE;
    if (chunk_cols < 1) return CCI_ERR_SHAPE;
    const bool tc_fits = Cin < (int64_t(1) << 31) && Cout < (int64_t(1) << 31);
    if (!tc_fits || !dense_tc_shape_ok(dtype, G, K, Cin, Cin)) return CCI_ERR_UNSUPPORTED;
    HostLayout l;
    if (!host_layout(dtype, Cin, Cout, chunk_cols, &l)) return CCI_ERR_SHAPE;
    if (!device_buffer || device_buffer_bytes < l.total || !aligned(device_buffer, 256)) return CCI_ERR_WORKSPACE;
    if (N == 0) return CCI_OK;

    const cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
    // the fused family multiplies every chunk from the packed weights (no
    // decompression); otherwise the first chunk decompresses into the workspace
    // and every chunk runs the workspace GEMM
    FwdParams probe = linear_params(device_buffer, 1, Cin, values, idx, Cout, static_cast<float *>(device_buffer),
                                    dev_status);
    probe.G = G;
    probe.K = K;
    const bool fused = auto_prefers_fused(K) && fused_may(probe, dtype) && gemm_pk_supported(probe);
    const cudaStream_t si = copy_in_stream ? reinterpret_cast<cudaStream_t>(copy_in_stream) : cs;
    const cudaStream_t so = copy_out_stream ? reinterpret_cast<cudaStream_t>(copy_out_stream) : cs;
    // events: [0] the call's start on `stream`; per slot k: chunk in (1 + k),
    // product done (1 + S + k), chunk out (1 + 2S + k)
    constexpr int kEv = 1 + 3 * kHostSlots;
    cudaEvent_t ev[kEv] = {};
    for (int i = 0; i < kEv; ++i) {
        if (cudaEventCreateWithFlags(&ev[i], cudaEventDisableTiming) != cudaSuccess) {
            for (int j = 0; j < i; ++j) cudaEventDestroy(ev[j]);
            return CCI_ERR_CUDA;
        }
    }
    cudaEvent_t *ev_in = ev + 1, *ev_done = ev + 1 + kHostSlots, *ev_out = ev + 1 + 2 * kHostSlots;
    char *const base = static_cast<char *>(device_buffer);
    void *const ws = base;
    char *const xs = base + l.ws;
    char *const ys = xs + kHostSlots * l.xslot;
    const size_t es = elem_size(dtype);
    const int64_t chunks = (N + chunk_cols - 1) / chunk_cols;

    // the copy streams start after the work the caller enqueued on `stream` before this call
    cudaError_t e = cudaEventRecord(ev[0], cs);
    if (e == cudaSuccess && si != cs) e = cudaStreamWaitEvent(si, ev[0], 0);
    if (e == cudaSuccess && so != cs) e = cudaStreamWaitEvent(so, ev[0], 0);
    cci_status result = to_status(e);
    int64_t issued = 0;  // chunks whose copy-out was enqueued
    for (int64_t c = 0; c < chunks && result == CCI_OK; ++c) {
        const int k = static_cast<int>(c % kHostSlots);
        const int64_t n0 = c * chunk_cols;
        const int64_t nc = (N - n0) < chunk_cols ? (N - n0) : chunk_cols;
        char *const xd = xs + k * l.xslot;
        float *const yd = reinterpret_cast<float *>(ys + k * l.yslot);
        // copy in, once the product of the chunk that last used this slot has read it
        if (c >= kHostSlots) e = cudaStreamWaitEvent(si, ev_done[k], 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(xd, static_cast<const char *>(X_host) + static_cast<size_t>(n0) * Cin * es,
                                static_cast<size_t>(nc) * Cin * es, cudaMemcpyHostToDevice, si);
        if (e == cudaSuccess) e = cudaEventRecord(ev_in[k], si);
        // product, once the chunk is in and the copy-out of this slot's last output is done
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ev_in[k], 0);
        if (e == cudaSuccess && c >= kHostSlots) e = cudaStreamWaitEvent(cs, ev_out[k], 0);
        result = to_status(e);
        if (result != CCI_OK) break;
        FwdParams p = linear_params(xd, nc, Cin, values, idx, Cout, yd, dev_status);
        p.G = G;
        p.K = K;
        if (fused) {
            result = to_status(launch_gemm_pk(p, cs));
        } else if (c == 0) {
            // the first chunk decompresses the weights into the workspace
            result = forward(p, dtype, G, K, CCI_ALGO_DENSE_TC_WS, ws, l.ws, cs);
        } else {
            p.wdense = ws;
            result = to_status(launch_gemm_ws(p, dtype, cs));
        }
        if (result != CCI_OK) break;
        e = cudaEventRecord(ev_done[k], cs);
        // copy out, once the product is done
        if (e == cudaSuccess) e = cudaStreamWaitEvent(so, ev_done[k], 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(Y_host + static_cast<size_t>(n0) * Cout, yd, static_cast<size_t>(nc) * Cout * 4,
                                cudaMemcpyDeviceToHost, so);
        if (e == cudaSuccess) e = cudaEventRecord(ev_out[k], so);
        result = to_status(e);
        if (result == CCI_OK) issued = c + 1;
    }
    // the call completes on `stream`: it waits for every copy-out enqueued
    for (int k = 0; k < kHostSlots && k < issued; ++k) {
        const cudaError_t w = cudaStreamWaitEvent(cs, ev_out[k], 0);
        if (result == CCI_OK) result = to_status(w);
    }
    for (int i = 0; i < kEv; ++i) cudaEventDestroy(ev[i]);  // released once their last record completes
    return result;
}
