// cci_gemm_ws.cu -- the dense tensor-core product of the workspace family
// (CCI_ALGO_DENSE_TC_WS) after the one-pass decompression of the packed weights.
//
// D[n][co] = sum_r x[n][r] * Wd[co][r] on tcgen05 with fp32 accumulators in TMEM:
//   bf16:  A = activation tile [128 n][64 r], B = weight tile [256 co][64 r], one
//          kind::f16 MMA per 16 r; 4 stages of 48 KB; two 256-column accumulators.
//   tf32x3 (fp32 layers): every operand split as hi + lo (hi: the low 13 mantissa
//          bits cleared, exactly a tf32 value; lo = x - hi exactly); per 8 r three
//          kind::tf32 MMAs lo*hi + hi*lo + hi*hi; tile [128 n][128 co][32 r],
//          3 stages of 64 KB (A hi, A lo, B hi, B lo); two 128-column accumulators.
// Operands (all K-major, 128-byte swizzle, 1024-byte aligned stage buffers):
//   weights    TMA from the workspace planes (tensor maps over [Cout][R]);
//   activations TMA over X[N][Cin] for bf16 products; otherwise the producer warps
//          gather them (cp.async for bf16 convolutions; registers, two stages
//          ahead, then the hi/lo split, for tf32x3).
// Roles: warps 0-3 epilogue (TMEM lanes), warps 4-7 producers of the activation
// planes that are not copied by TMA, warp 8 allocates TMEM and issues the MMAs,
// warp 9 issues the TMA copies as soon as a stage is free (so copy latency
// overlaps the producers' work).  Every mbarrier wait is bounded
// (CCI_ERR_TIMEOUT, abort flag, drain, TMEM freed).
#include <cuda.h>
#include <cudaTypedefs.h>

#include "cci_tc_common.cuh"

namespace cci {
namespace ws {

enum Mode { kBf16Tma = 0, kBf16Gather = 1, kTf32x3 = 2, kTf32x3Tma = 3 };

template <int MODE>
struct Cfg;
template <>
struct Cfg<kBf16Tma> {
    static constexpr int kM = 128, kN = 256, kKS = 64, kStages = 4, kAPlanes = 1, kBPlanes = 1;
    static constexpr bool kATma = true, kTf32 = false;
};
template <>
struct Cfg<kBf16Gather> {
    static constexpr int kM = 128, kN = 256, kKS = 64, kStages = 4, kAPlanes = 1, kBPlanes = 1;
    static constexpr bool kATma = false, kTf32 = false;
};
template <>
struct Cfg<kTf32x3> {  // convolutions: activations gathered through registers
    static constexpr int kM = 128, kN = 128, kKS = 32, kStages = 3, kAPlanes = 2, kBPlanes = 2;
    static constexpr bool kATma = false, kTf32 = true;
};
template <>
struct Cfg<kTf32x3Tma> {  // products: the raw activation tile by TMA, split in shared memory
    static constexpr int kM = 128, kN = 128, kKS = 32, kStages = 3, kAPlanes = 2, kBPlanes = 2;
    static constexpr bool kATma = false, kTf32 = true;
};

template <int MODE>
struct Geo {
    using C = Cfg<MODE>;
    static constexpr int kAPlane = C::kM * 128;  // bytes: 128-byte rows
    static constexpr int kBPlane = C::kN * 128;
    static constexpr int kStage = C::kAPlanes * kAPlane + C::kBPlanes * kBPlane;
    static constexpr int kTmemCols = 2 * C::kN;
    static constexpr size_t kSmem = 1024 + static_cast<size_t>(C::kStages) * kStage + sizeof(tc::Smem) + 64;
    static constexpr uint32_t kTxBytes = (C::kATma ? C::kAPlanes * kAPlane : 0) + C::kBPlanes * kBPlane;
    static constexpr uint32_t kIdesc = (1u << 4)                                             // D f32
                                       | (C::kTf32 ? (2u << 7) | (2u << 10) : (1u << 7) | (1u << 10))  // tf32 / bf16
                                       | (static_cast<uint32_t>(C::kN >> 3) << 17) |
                                       (static_cast<uint32_t>(C::kM >> 4) << 24);
    static_assert(kSmem <= kMaxSmemPerBlock, "stage buffers over the per-block limit");
};

template <int MODE>
__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t acc)
{
    if constexpr (Cfg<MODE>::kTf32) {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(a), "l"(b), "r"(Geo<MODE>::kIdesc), "r"(acc)
            : "memory");
    } else {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(a), "l"(b), "r"(Geo<MODE>::kIdesc), "r"(acc)
            : "memory");
    }
}

// byte offset of (row, 16-byte chunk) in a plane of 128-byte rows, 128-byte swizzle
__device__ __forceinline__ uint32_t sw_chunk(int row, int chunk)
{
    return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) * 16));
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ uint32_t hi_bits(uint32_t x) { return x & 0xffffe000u; }
__device__ __forceinline__ uint32_t lo_bits(uint32_t x)
{
    return __float_as_uint(__uint_as_float(x) - __uint_as_float(hi_bits(x)));
}

constexpr int kThreads = 320;

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_ws_kernel(FwdParams p, const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
                   const __grid_constant__ CUtensorMap tmB1, int64_t n_ct, int64_t n_tiles)
{
    using C = Cfg<MODE>;
    using GE = Geo<MODE>;
    constexpr int kM = C::kM, kN = C::kN, kKS = C::kKS, kStages = C::kStages;
    constexpr int kLag = 2;  // bf16 gather: stages in flight before a producer's arrive
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t raw = tc::smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    tc::Smem *S = reinterpret_cast<tc::Smem *>(smem_raw + (base - raw) + kStages * GE::kStage);
    volatile int *abort = &S->abort;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nks = static_cast<int>((p.R + kKS - 1) / kKS);

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&S->full[s], C::kATma ? 1 : 129);
            tc::mbar_init(&S->empty[s], 1);
            tc::mbar_init(&S->aux[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            tc::mbar_init(&S->tmem_full[a], 1);
            tc::mbar_init(&S->tmem_empty[a], 128);
        }
        tc::mbar_init(&S->drain, 1);
        S->abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 8) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         tc::smem_u32(&S->tmem_base)),
                     "r"(GE::kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid == 288) {
        if constexpr (C::kATma || MODE == kTf32x3Tma) tc::tma_prefetch_desc(&tmA);
        tc::tma_prefetch_desc(&tmB0);
        if constexpr (C::kBPlanes > 1) tc::tma_prefetch_desc(&tmB1);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = S->tmem_base;

    if (warp == 9) {
        // ------------------------------------------------------------ TMA issuer
        int it = 0;
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
            const int64_t n0 = (tile / n_ct) * kM;
            const int64_t co0 = (tile % n_ct) * kN;
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                if (it >= kStages) ok = tc::mbar_wait(&S->empty[s], ((it / kStages) - 1) & 1, abort, p.status);
                if (!ok) break;
                if (lane == 0) {
                    const uint32_t st = base + s * GE::kStage;
                    const uint32_t bst = st + C::kAPlanes * GE::kAPlane;
                    if constexpr (MODE == kTf32x3Tma) {
                        tc::mbar_arrive_expect_tx(&S->aux[s], GE::kAPlane);
                        tc::tma_load_2d(st, &tmA, ks * kKS, static_cast<int>(n0), &S->aux[s]);
                    }
                    tc::mbar_arrive_expect_tx(&S->full[s], GE::kTxBytes);
                    tc::tma_load_2d(bst, &tmB0, ks * kKS, static_cast<int>(co0), &S->full[s]);
                    if constexpr (C::kBPlanes > 1)
                        tc::tma_load_2d(bst + GE::kBPlane, &tmB1, ks * kKS, static_cast<int>(co0), &S->full[s]);
                    if constexpr (C::kATma) tc::tma_load_2d(st, &tmA, ks * kKS, static_cast<int>(n0), &S->full[s]);
                }
                __syncwarp();
            }
        }
    } else if (warp >= 4 && warp < 8) {
        // ------------------------------------------------------------ producers
        const int pt = tid - 128;
        const int chunk = pt & 7;  // 16-byte chunk of every activation row this thread gathers
        const int rowb = pt >> 3;  // rows rowb + 16 i
        int it = 0;
        bool ok = true;
        // tf32x3: activation chunks of the next two stages, in registers
        uint4 xa[8], xb[8], xc[8];
        ColumnSite xsite[8];  // column sites of the tile being prefetched
        int64_t xsite_tile = -1;
        auto load_x = [&](uint4 (&dst)[8], int64_t tile, int ks) {
#pragma unroll
            for (int i = 0; i < 8; ++i) dst[i] = make_uint4(0, 0, 0, 0);
            if (tile >= n_tiles || ks >= nks) return;
            const int64_t n0 = (tile / n_ct) * kM;
            if (tile != xsite_tile) {
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int64_t n = n0 + rowb + 16 * i;
                    xsite[i] = n < p.N ? column_site(p, n) : ColumnSite{-1, 0, 0};
                }
                xsite_tile = tile;
            }
            const int64_t r = static_cast<int64_t>(ks) * kKS + chunk * 4;
            if (r >= p.R) return;
            int kh = 0, kw = 0;
            int64_t ci = r;
            if (p.is_conv) {
                const int tap = static_cast<int>(r / p.Cin);
                ci = r - static_cast<int64_t>(tap) * p.Cin;
                kh = tap / p.KW;
                kw = tap - kh * p.KW;
            }
            const float *X = static_cast<const float *>(p.X);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (xsite[i].img < 0) continue;  // column past N
                int64_t off = xsite[i].img + r;
                if (p.is_conv) {
                    const int h = xsite[i].hb + kh, w = xsite[i].wb + kw;
                    if (h < 0 || h >= p.H || w < 0 || w >= p.W) continue;
                    off = xsite[i].img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
                }
                dst[i] = __ldg(reinterpret_cast<const uint4 *>(X + off));
            }
        };
        // (tile, ks) of the stage `ahead` stages after (tile, ks)
        auto advance = [&](int64_t &tile, int &ks) {
            if (++ks == nks) {
                ks = 0;
                tile += gridDim.x;
            }
        };
        int64_t t1 = blockIdx.x, t2 = blockIdx.x;
        int k1 = 0, k2 = 0;
        if constexpr (MODE == kTf32x3) {
            load_x(xa, t1, k1);
            advance(t2, k2);
            load_x(xb, t2, k2);
            advance(t2, k2);
        }
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
            const int64_t ct = tile % n_ct;
            const int64_t n0 = (tile / n_ct) * kM;
            const int64_t co0 = ct * kN;
            ColumnSite site[8];
            bool colok[8];
            if constexpr (MODE == kBf16Gather) {
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int64_t n = n0 + rowb + 16 * i;
                    colok[i] = n < p.N;
                    site[i] = colok[i] ? column_site(p, n) : ColumnSite{0, 0, 0};
                }
            }
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                if constexpr (MODE == kTf32x3) load_x(xc, t2, k2);  // two stages ahead
                // gather / register modes write the stage themselves: wait until it is
                // free; the split mode waits for its raw tile (copied after the stage
                // was freed) instead
                if (MODE != kTf32x3Tma && it >= kStages)
                    ok = tc::mbar_wait(&S->empty[s], ((it / kStages) - 1) & 1, abort, p.status);
                if (!ok) break;
                const uint32_t st = base + s * GE::kStage;
                if constexpr (MODE == kBf16Gather) {
                    const uint16_t *X = static_cast<const uint16_t *>(p.X);
                    const int64_t r = static_cast<int64_t>(ks) * kKS + chunk * 8;
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
                        tc::cp_async16(st + sw_chunk(rowb + 16 * i, chunk), src, valid);
                    }
                    asm volatile("cp.async.commit_group;" ::: "memory");
                    if (it >= kLag) {
                        asm volatile("cp.async.wait_group %0;" ::"n"(kLag) : "memory");
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        tc::mbar_arrive(&S->full[(it - kLag) % kStages]);
                    }
                } else if constexpr (MODE == kTf32x3Tma) {
                    // the raw fp32 tile landed in the hi plane: split it in place
                    ok = tc::mbar_wait(&S->aux[s], (it / kStages) & 1, abort, p.status);
                    if (!ok) break;
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const uint32_t o = sw_chunk(rowb + 16 * i, chunk);
                        uint4 v;
                        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                                     : "r"(st + o)
                                     : "memory");
                        st_shared_v4(st + o, hi_bits(v.x), hi_bits(v.y), hi_bits(v.z), hi_bits(v.w));
                        st_shared_v4(st + GE::kAPlane + o, lo_bits(v.x), lo_bits(v.y), lo_bits(v.z), lo_bits(v.w));
                    }
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    tc::mbar_arrive(&S->full[s]);
                } else if constexpr (C::kTf32) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const uint32_t o = sw_chunk(rowb + 16 * i, chunk);
                        st_shared_v4(st + o, hi_bits(xa[i].x), hi_bits(xa[i].y), hi_bits(xa[i].z), hi_bits(xa[i].w));
                        st_shared_v4(st + GE::kAPlane + o, lo_bits(xa[i].x), lo_bits(xa[i].y), lo_bits(xa[i].z),
                                     lo_bits(xa[i].w));
                    }
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    tc::mbar_arrive(&S->full[s]);
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        xa[i] = xb[i];
                        xb[i] = xc[i];
                    }
                    advance(t2, k2);
                }
            }
        }
        if constexpr (MODE == kBf16Gather) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            for (int q = (it >= kLag ? it - kLag : 0); q < it; ++q) tc::mbar_arrive(&S->full[q % kStages]);
        }
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        int it = 0, t = 0;
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
            const int acc = t & 1;
            if (t >= 2) ok = tc::mbar_wait(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                ok = tc::mbar_wait(&S->full[s], (it / kStages) & 1, abort, p.status);
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                if (lane == 0) {
                    const uint32_t st = base + s * GE::kStage;
                    const uint32_t bst = st + C::kAPlanes * GE::kAPlane;
                    if constexpr (C::kTf32) {
#pragma unroll
                        for (int k = 0; k < kKS / 8; ++k) {
                            const uint64_t ah = tc::sw128_desc(st + k * 32);
                            const uint64_t al = tc::sw128_desc(st + GE::kAPlane + k * 32);
                            const uint64_t bh = tc::sw128_desc(bst + k * 32);
                            const uint64_t bl = tc::sw128_desc(bst + GE::kBPlane + k * 32);
                            mma<MODE>(d, al, bh, (ks > 0 || k > 0) ? 1u : 0u);
                            mma<MODE>(d, ah, bl, 1u);
                            mma<MODE>(d, ah, bh, 1u);
                        }
                    } else {
#pragma unroll
                        for (int k = 0; k < kKS / 16; ++k)
                            mma<MODE>(d, tc::sw128_desc(st + k * 32), tc::sw128_desc(bst + k * 32),
                                      (ks > 0 || k > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(&S->empty[s]);
                }
                __syncwarp();
            }
            if (ok && lane == 0) tc::mma_commit(&S->tmem_full[acc]);
            __syncwarp();
        }
        if (lane == 0) tc::mma_commit(&S->drain);
        __syncwarp();
        int no_abort = 0;
        tc::mbar_wait(&S->drain, 0, &no_abort, p.status);
    } else {
        // ------------------------------------------------------------ epilogue (warps 0-3)
        int t = 0;
        bool ok = true;
        const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
        for (int64_t tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++t) {
            const int acc = t & 1;
            const int64_t ct = tile % n_ct;
            const int64_t n0 = (tile / n_ct) * kM;
            ok = tc::mbar_wait(&S->tmem_full[acc], (t / 2) & 1, abort, p.status);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int64_t n = n0 + warp * 32 + lane;
            const int64_t co0 = ct * kN;
#pragma unroll 1
            for (int c = 0; c < kN / 32; ++c) {
                uint32_t v[32];
                tc::tmem_ld32(tmem + lane_off + static_cast<uint32_t>(acc * kN + c * 32), v);
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
            tc::mbar_arrive(&S->tmem_empty[acc]);
        }
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 8) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(GE::kTmemCols)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------
// host: tensor maps and launch
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }();
    return fn;
}

// 2-D map over a row-major [rows][inner] array, box [box_rows][box_inner], 128-byte swizzle
bool make_map(CUtensorMap *m, const void *ptr, CUtensorMapDataType dt, int elem, int64_t inner, int64_t rows,
              int box_inner, int box_rows)
{
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(inner) * elem};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_rows)};
    cuuint32_t es[2] = {1, 1};
    return fn(m, dt, 2, const_cast<void *>(ptr), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int MODE>
cudaError_t launch_mode(const FwdParams &p, cudaStream_t stream)
{
    using C = Cfg<MODE>;
    using GE = Geo<MODE>;
    auto kern = gemm_ws_kernel<MODE>;
    static const cudaError_t attr =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(GE::kSmem));
    if (attr != cudaSuccess) return attr;
    CUtensorMap tmA{}, tmB0{}, tmB1{};
    const CUtensorMapDataType dt = C::kTf32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int elem = C::kTf32 ? 4 : 2;
    if ((C::kATma || MODE == kTf32x3Tma) && !make_map(&tmA, p.X, dt, elem, p.Cin, p.N, C::kKS, C::kM))
        return cudaErrorInvalidValue;
    if (!make_map(&tmB0, p.wdense, dt, elem, p.R, p.Cout, C::kKS, C::kN)) return cudaErrorInvalidValue;
    if (C::kBPlanes > 1) {
        const char *lo = static_cast<const char *>(p.wdense) + static_cast<size_t>(p.Cout) * p.R * elem;
        if (!make_map(&tmB1, lo, dt, elem, p.R, p.Cout, C::kKS, C::kN)) return cudaErrorInvalidValue;
    }
    const int64_t n_ct = (p.Cout + C::kN - 1) / C::kN;
    const int64_t n_tiles = n_ct * ((p.N + C::kM - 1) / C::kM);
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t grid = n_tiles < sms ? n_tiles : sms;
    kern<<<static_cast<unsigned>(grid), kThreads, GE::kSmem, stream>>>(p, tmA, tmB0, tmB1, n_ct, n_tiles);
    return cudaGetLastError();
}

}  // namespace ws

cudaError_t launch_gemm_ws(const FwdParams &p, int dtype, cudaStream_t stream)
{
    if (dtype == CCI_F32) return p.is_conv ? ws::launch_mode<ws::kTf32x3>(p, stream)
                                           : ws::launch_mode<ws::kTf32x3Tma>(p, stream);
    if (!p.is_conv) return ws::launch_mode<ws::kBf16Tma>(p, stream);
    return ws::launch_mode<ws::kBf16Gather>(p, stream);
}

}  // namespace cci
