// cci_dense_tc.cu -- comparison kernel: decompress the packed weights to dense
// bf16 tiles in shared memory and multiply them on the tensor cores (tcgen05);
// and the one-pass decompression into the workspace of CCI_ALGO_DENSE_TC_WS
// (namespace dc) that precedes the workspace GEMM.
//
// The product of Alg. 2 equals the dense product with the pruned weights zero
// (Sec. 3.1); this kernel computes it densely, paying G/K times the useful
// multiply-adds at tensor-core rate instead of the index dispatch on CUDA cores.
//
// Tile: D[128 columns n][256 channels co] fp32 in TMEM (two accumulator
// buffers of 256 columns), K = 64 reduction indices per pipeline stage.
//   A = activation tile [128 n][64 r] bf16, K-major, 128-byte swizzle
//   B = weight tile     [256 co][64 r] bf16, K-major, 128-byte swizzle
// Warp roles (288 threads):
//   warps 0-3  epilogue: tcgen05.ld of TMEM lanes 32*w.. (column n = lane), fp32 rows
//              of Y[n][co] stored as float4;
//   warps 4-7  producers: cp.async gather of the activation rows (product or
//              implicit convolution, zero outside the image / past N) straight into
//              the swizzled layout, and decompression of the CTA's packed groups
//              (zero the group's rows, then write its K values per r);
//   warp 8     allocates TMEM and issues tcgen05.mma (one elected lane).
// Every mbarrier wait is bounded: on expiry the kernel records CCI_ERR_TIMEOUT,
// raises a CTA abort flag so the other roles stop, drains its own copies and
// MMAs, frees TMEM and exits.
#include "cci_tc_common.cuh"

namespace cci {
namespace tc {

constexpr int kM = 128;       // columns per tile (MMA M)
constexpr int kN = 256;       // channels per tile (MMA N)
constexpr int kKS = 64;       // reduction indices per stage (128 bytes of bf16)
constexpr int kStages = 4;
constexpr int kLag = 2;       // producer stages in flight before their arrive
constexpr int kThreads = 288;
constexpr int kATile = kM * kKS * 2;   // 16 KB
constexpr int kBTile = kN * kKS * 2;   // 32 KB
constexpr int kTmemCols = 512;         // two 256-column fp32 accumulators

constexpr size_t kSmemBytes = 1024 /*alignment slack*/ + kStages * (kATile + kBTile) + sizeof(Smem) + 64;

// instruction descriptor, kind::f16: D f32, A and B bf16, both K-major, M x N
constexpr uint32_t kIdesc = (1u << 4)                 // D format f32
                            | (1u << 7) | (1u << 10)  // A, B format bf16
                            | (static_cast<uint32_t>(kN >> 3) << 17) | (static_cast<uint32_t>(kM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate)
{
    asm volatile(
        "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}


template <int G, int K, bool WS>
__global__ void __launch_bounds__(kThreads, 1) dense_tc_kernel(FwdParams p, int64_t n_ct, int64_t n_tiles)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;  // 1024-byte aligned stage area
    unsigned char *gbase = smem_raw + (base - raw);
    Smem *S = reinterpret_cast<Smem *>(gbase + kStages * (kATile + kBTile));
    const uint32_t a_smem = base;                            // stages of A
    const uint32_t b_smem = base + kStages * kATile;         // stages of B
    volatile int *abort = &S->abort;

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int64_t total_groups = p.Cout / G;
    const int nks = static_cast<int>((p.R + kKS - 1) / kKS);
    const uint16_t *X = static_cast<const uint16_t *>(p.X);
    const uint16_t *V = static_cast<const uint16_t *>(p.values);

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&S->full[s], 128);
            mbar_init(&S->empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&S->tmem_full[a], 1);
            mbar_init(&S->tmem_empty[a], 128);
        }
        mbar_init(&S->drain, 1);
        S->abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 8) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&S->tmem_base)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = S->tmem_base;

    if (warp >= 4 && warp < 8) {
        // ------------------------------------------------------------ producers
        const int pt = tid - 128;
        const int chunk = pt & 7;  // 16-byte chunk (8 indices) of every copy this thread makes
        const int rowb = pt >> 3;  // rows rowb + 16 * i, i < 8
        int it = 0;                // stage counter of this CTA
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
            const int64_t ct = tile % n_ct;
            const int64_t n0 = (tile / n_ct) * kM;
            const int64_t g0 = ct * (kN / G);
            ColumnSite site[8];
            bool colok[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int64_t n = n0 + rowb + 16 * i;
                colok[i] = n < p.N;
                site[i] = colok[i] ? column_site(p, n) : ColumnSite{0, 0, 0};
            }
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                if (it >= kStages) ok = mbar_wait(&S->empty[s], ((it / kStages) - 1) & 1, abort, p.status);
                if (!ok) break;
                const int64_t r0 = static_cast<int64_t>(ks) * kKS;
                // A: 128 rows x 8 chunks of 16 bytes; this thread: chunk `chunk` of 8 rows
                const int64_t r = r0 + chunk * 8;
                const bool rok = r < p.R;
                int kh = 0, kw = 0;
                int64_t ci = r;
                if (p.is_conv && rok) {
                    const int tap = static_cast<int>(r / p.Cin);
                    ci = r - static_cast<int64_t>(tap) * p.Cin;
                    kh = tap / p.KW;
                    kw = tap - kh * p.KW;
                }
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int row = rowb + 16 * i;
                    bool valid = colok[i] && rok;
                    const uint16_t *src = X;
                    if (valid) {
                        if (!p.is_conv) {
                            src = X + site[i].img + r;
                        } else {
                            const int h = site[i].hb + kh, w = site[i].wb + kw;
                            valid = h >= 0 && h < p.H && w >= 0 && w < p.W;
                            if (valid) src = X + site[i].img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
                        }
                    }
                    cp_async16(a_smem + s * kATile + sw128(row, chunk * 8), src, valid);
                }
                const uint32_t bt = b_smem + s * kBTile;
                if constexpr (WS) {
                    // B: 256 rows x 8 chunks of the dense weights; rows rowb + 16 i, chunk `chunk`
                    const uint16_t *Wd = static_cast<const uint16_t *>(p.wdense);
                    const int64_t co0 = ct * kN;
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int row = rowb + 16 * i;
                        const bool valid = co0 + row < p.Cout && rok;
                        cp_async16(bt + sw128(row, chunk * 8), valid ? Wd + (co0 + row) * p.R + r : Wd, valid);
                    }
                }
                asm volatile("cp.async.commit_group;" ::: "memory");
                if constexpr (!WS) {
                // B: units (group, 8-index chunk): zero the group's G rows of the
                // chunk, then write the K kept values of each of the 8 indices
                for (int u = pt; u < (kN / G) * 8; u += 128) {
                    const int gl = u >> 3, chunk = u & 7;
#pragma unroll
                    for (int j = 0; j < G; ++j) st_shared_v4_zero(bt + static_cast<uint32_t>((gl * G + j) * 128 + ((chunk ^ ((gl * G + j) & 7)) * 16)));
                    const int64_t gg = g0 + gl;
                    if (gg >= total_groups) continue;
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int64_t r = r0 + chunk * 8 + e;
                        if (r >= p.R) break;
                        const int64_t o = (gg * p.R + r) * K;
                        int prev = -1;
#pragma unroll
                        for (int sl = 0; sl < K; ++sl) {
                            const int i = __ldg(p.idx + o + sl);
                            if (i >= G || i <= prev) {  // index sets must be strictly increasing
                                report(p.status, CCI_ERR_INDEX);
                                continue;
                            }
                            prev = i;
                            const uint16_t val = __ldg(V + o + sl);
                            st_shared_b16(bt + sw128(gl * G + i, chunk * 8 + e), val);
                        }
                    }
                }
                }
                // stage it - kLag is complete for this thread: its copies landed
                if (it >= kLag) {
                    asm volatile("cp.async.wait_group %0;" ::"n"(kLag) : "memory");
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    mbar_arrive(&S->full[(it - kLag) % kStages]);
                }
            }
        }
        // flush: arrive for the last stages still pending
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        for (int q = (it >= kLag ? it - kLag : 0); q < it; ++q) mbar_arrive(&S->full[q % kStages]);
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        int it = 0, t = 0;
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
            const int acc = t & 1;
            if (t >= 2) ok = mbar_wait(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                ok = mbar_wait(&S->full[s], (it / kStages) & 1, abort, p.status);
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                if (lane == 0) {
#pragma unroll
                    for (int k = 0; k < kKS / 16; ++k) {
                        const uint64_t ad = sw128_desc(a_smem + s * kATile + k * 32);
                        const uint64_t bd = sw128_desc(b_smem + s * kBTile + k * 32);
                        mma_bf16(d, ad, bd, (ks > 0 || k > 0) ? 1u : 0u);
                    }
                    mma_commit(&S->empty[s]);
                }
                __syncwarp();
            }
            if (ok && lane == 0) mma_commit(&S->tmem_full[acc]);
            __syncwarp();
        }
        // drain: every MMA issued by this thread has completed before TMEM is freed
        if (lane == 0) mma_commit(&S->drain);
        __syncwarp();
        int dummy_abort = 0;
        mbar_wait(&S->drain, 0, &dummy_abort, p.status);
    } else {
        // ------------------------------------------------------------ epilogue (warps 0-3)
        int t = 0;
        bool ok = true;
        const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
            const int acc = t & 1;
            const int64_t ct = tile % n_ct;
            const int64_t n0 = (tile / n_ct) * kM;
            ok = mbar_wait(&S->tmem_full[acc], (t / 2) & 1, abort, p.status);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int64_t n = n0 + warp * 32 + lane;
            const int64_t co0 = ct * kN;
#pragma unroll 1
            for (int c = 0; c < kN / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_off + static_cast<uint32_t>(acc * kN + c * 32), v);
                if (n < p.N) {
                    float *y = p.Y + n * p.Cout + co0 + c * 32;
                    if (co0 + c * 32 + 32 <= p.Cout) {
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            __stcs(reinterpret_cast<float4 *>(y) + q,
                                   make_float4(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]),
                                               __uint_as_float(v[4 * q + 2]), __uint_as_float(v[4 * q + 3])));
                    } else {
                        for (int q = 0; q < 32 && co0 + c * 32 + q < p.Cout; ++q) y[q] = __uint_as_float(v[q]);
                    }
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            mbar_arrive(&S->tmem_empty[acc]);
        }
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 8) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

template <int G, int K, bool WS>
cudaError_t launch(const FwdParams &p, cudaStream_t stream)
{
    auto kern = dense_tc_kernel<G, K, WS>;
    static SmemAttrCache attr_cache;
    const cudaError_t attr = smem_attr_once(kern, static_cast<int>(kSmemBytes), attr_cache);
    if (attr != cudaSuccess) return attr;
    const int64_t n_ct = (p.Cout + kN - 1) / kN;
    const int64_t n_nt = (p.N + kM - 1) / kM;
    const int64_t n_tiles = n_ct * n_nt;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = n_tiles < sms ? n_tiles : sms;
    kern<<<static_cast<unsigned>(grid), kThreads, kSmemBytes, stream>>>(p, n_ct, n_tiles);
    return cudaGetLastError();
}

// Diagnostic of the bounded waits above: one thread initialises an mbarrier that
// expects one arrival, arrives on it when `arrive` is set, and waits for its
// phase with mbar_wait.  Without the arrival nothing can complete the phase, the
// wait gives up after kWaitLimit cycles and reports CCI_ERR_TIMEOUT; nothing is
// in flight, so the kernel then simply returns.
__global__ void wait_probe_kernel(uint32_t *status, int arrive)
{
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        if (arrive) mbar_arrive(&bar);
        mbar_wait(&bar, 0, &abort_flag, status);
    }
}

}  // namespace tc

cudaError_t launch_wait_probe(uint32_t *status, int arrive, cudaStream_t stream)
{
    tc::wait_probe_kernel<<<1, 32, 0, stream>>>(status, arrive);
    return cudaGetLastError();
}

// ===========================================================================
// One-pass decompression of the packed weights into the workspace of
// CCI_ALGO_DENSE_TC_WS: the dense W[Cout][R] (bf16, bit for bit), or for fp32
// layers its hi and lo tf32 planes [2][Cout][R] (hi = w with the low 13 mantissa
// bits cleared, exactly a tf32 value; lo = w - hi, exact in fp32) for the
// three-pass product hi*hi + hi*lo + lo*hi.
// One block per (group gi, slab of kSlab columns r): each thread scatters the K
// kept weights of one column into a zeroed [G][kSlab] tile in shared memory,
// then the block writes the G rows of the slab with 16-byte stores.  Index sets
// must be strictly increasing (as cci_pack writes them); anything else is
// reported as CCI_ERR_INDEX.
// ===========================================================================
namespace dc {

constexpr int kSlab = 256;  // columns r per block (= threads per block)

__device__ __forceinline__ uint32_t hi_bits(uint32_t x) { return x & 0xffffe000u; }
__device__ __forceinline__ uint32_t lo_bits(uint32_t x)
{
    return __float_as_uint(__uint_as_float(x) - __uint_as_float(hi_bits(x)));
}

// T = uint16_t (bf16 bits) or uint32_t (fp32 bits); SPLIT: write hi to w0 and
// lo to w1 (fp32 only), else the weights to w0.  R must be a multiple of the
// elements per 16 bytes.
template <typename T, int G, int K, bool SPLIT>
__global__ void __launch_bounds__(kSlab) decompress_kernel(const T *__restrict__ values,
                                                           const uint8_t *__restrict__ idx, int64_t R,
                                                           int64_t slabs, T *__restrict__ w0, T *__restrict__ w1,
                                                           uint32_t *status)
{
    constexpr int V = 16 / static_cast<int>(sizeof(T));  // elements per 16-byte store
    __shared__ __align__(16) T tile[G][kSlab];
    // the workspace GEMM that follows may start its prologue now; it waits for
    // this grid's completion before reading the workspace
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t gi = blockIdx.x / slabs;
    const int64_t r0 = (blockIdx.x - gi * slabs) * kSlab;
    for (int e = threadIdx.x; e < G * kSlab / V; e += kSlab)
        reinterpret_cast<uint4 *>(&tile[0][0])[e] = make_uint4(0, 0, 0, 0);
    __syncthreads();
    const int64_t r = r0 + threadIdx.x;
    if (r < R) {
        const int64_t t = gi * R + r;
        bool bad = false;
        int prev = -1;
#pragma unroll
        for (int s = 0; s < K; ++s) {
            const T v = values[t * K + s];
            const int j = idx[t * K + s];
            bad |= j >= G || j <= prev;
            prev = j;
            if (j < G) tile[j][threadIdx.x] = v;
        }
        if (bad) report(status, CCI_ERR_INDEX);
    }
    __syncthreads();
    constexpr int kVecs = kSlab / V;  // 16-byte vectors per tile row
    for (int e = threadIdx.x; e < G * kVecs; e += kSlab) {
        const int j = e / kVecs, c = e - j * kVecs;
        const int64_t rr = r0 + static_cast<int64_t>(c) * V;
        if (rr >= R) continue;
        const uint4 x = *reinterpret_cast<const uint4 *>(&tile[j][c * V]);
        const int64_t off = (gi * G + j) * R + rr;
        if constexpr (SPLIT) {
            __stcg(reinterpret_cast<uint4 *>(w0 + off), make_uint4(hi_bits(x.x), hi_bits(x.y), hi_bits(x.z), hi_bits(x.w)));
            __stcg(reinterpret_cast<uint4 *>(w1 + off), make_uint4(lo_bits(x.x), lo_bits(x.y), lo_bits(x.z), lo_bits(x.w)));
        } else {
            __stcg(reinterpret_cast<uint4 *>(w0 + off), x);
        }
    }
}

template <typename T, int G, int K, bool SPLIT>
cudaError_t launch(const FwdParams &p, cudaStream_t stream)
{
    const int64_t slabs = (p.R + kSlab - 1) / kSlab;
    const int64_t blocks = (p.Cout / G) * slabs;
    if (blocks > 0x7fffffff) return cudaErrorInvalidValue;
    T *w0 = static_cast<T *>(const_cast<void *>(p.wdense));
    T *w1 = SPLIT ? w0 + p.Cout * p.R : nullptr;
    decompress_kernel<T, G, K, SPLIT><<<static_cast<unsigned>(blocks), kSlab, 0, stream>>>(
        static_cast<const T *>(p.values), p.idx, p.R, slabs, w0, w1, p.status);
    return cudaGetLastError();
}

}  // namespace dc

// (G, K) pairs with a dense tensor-core instantiation (G divides the 256-channel tile)
cudaError_t launch_dense_tc(const FwdParams &p, int dtype, int G, int K, bool ws, cudaStream_t stream)
{
    if (dtype == CCI_F32 && !ws) return cudaErrorNotSupported;
#define CCI_TC_CASE(g, k)                                                                   \
    if (G == g && K == k) {                                                                 \
        if (!ws) return tc::launch<g, k, false>(p, stream);                                 \
        const cudaError_t e = dtype == CCI_F32 ? dc::launch<uint32_t, g, k, true>(p, stream) \
                                               : dc::launch<uint16_t, g, k, false>(p, stream); \
        if (e != cudaSuccess) return e;                                                     \
        return launch_gemm_ws(p, dtype, stream);                                            \
    }
    CCI_TC_CASE(4, 1) CCI_TC_CASE(4, 2)
    CCI_TC_CASE(8, 1) CCI_TC_CASE(8, 2) CCI_TC_CASE(8, 4)
    CCI_TC_CASE(16, 1) CCI_TC_CASE(16, 2) CCI_TC_CASE(16, 4) CCI_TC_CASE(16, 8)
    CCI_TC_CASE(32, 1) CCI_TC_CASE(32, 2) CCI_TC_CASE(32, 4) CCI_TC_CASE(32, 8) CCI_TC_CASE(32, 16)
#undef CCI_TC_CASE
    return cudaErrorNotSupported;
}

bool dense_tc_supported(int dtype, int G, int K)
{
    if (dtype != CCI_BF16 && dtype != CCI_F32) return false;
    const int gs[] = {4, 8, 16, 32};
    for (int g : gs)
        if (g == G) return K >= 1 && K <= G / 2 && (K & (K - 1)) == 0;
    return false;
}

}  // namespace cci
