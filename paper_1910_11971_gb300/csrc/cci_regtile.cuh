// cci_regtile.cuh -- register-tiled CCI scatter kernel for sm_103a.
//
// Computes Alg. 2 of Sec. 3.2 (H(G*i + Idx, j) += Val * X(k, j), with a slot
// loop for K > 1) for a product or an implicit convolution.
//
// Work split (the group-boundary split of Sec. 3.2: a CTA owns whole groups):
//   * a CTA of 8 warps owns WC*MG whole groups (WC warps across channels, each
//     owning MG groups) and NTC = (8/WC)*32*T columns (8/WC warps across columns);
//   * lane l of a warp owns T columns: 4-column runs at l*4 + q*128, q < T/4;
//   * the index of a slot depends on (group, r, slot), not on the column, so all
//     lanes of a warp take the same index at the same time: the choice of the
//     output row in Alg. 2 is one warp-uniform jump (generated PTX brx.idx, see
//     cci_dispatch.cuh) into straight-line packed FMAs, and the MG*G x T block of
//     outputs stays in registers ("load a whole group of elements of H onto
//     on-chip registers", Sec. 3.2);
//   * two columns share one packed FMA (fma.rn.f32x2);
//   * expand mode (D = 0) takes no jump: each record holds the G weights of the
//     (group, r) with the pruned ones zero and the lane runs G straight-line
//     packed FMAs per column pair -- G/K times the useful work, but no
//     warp-uniform jumps, which cost far more than an FMA on this GPU.
//
// Pipeline per chunk of RC = 16 reduction indices:
//   raw X tile [NTC][RC] and raw (value, index) runs are copied global->shared
//   with cp.async one chunk ahead (no registers held); the chunk is then
//   transposed to an fp32 [RC][NTC] tile (bf16 widened exactly) and each
//   (group, r) gets a record of 16-byte units: K fp32 values, then the dispatch
//   words (D = 1: the indices, 4 per word; D = 2: per slot pair the colex rank
//   of the ascending pair in bits 0-7 and the raw indices in bits 8-23).
//   Per output channel the contributions arrive in ascending r (then slot), one
//   fused multiply-add each, starting from +0.
#pragma once

#include "cci_common.cuh"
#include "cci_dispatch.cuh"

namespace cci {

template <typename TS>
struct Elem;
template <>
struct Elem<float> {
    static constexpr int kVec = 4;  // elements per 16 bytes
    __device__ static float to_f32(float v) { return v; }
    __device__ static float widen(const uint32_t (&w)[4], int e) { return __uint_as_float(w[e]); }
};
template <>
struct Elem<uint16_t> {  // bfloat16 bits
    static constexpr int kVec = 8;
    __device__ static float to_f32(uint16_t v) { return bf16_bits_to_f32(v); }
    __device__ static float widen(const uint32_t (&w)[4], int e)
    {
        const uint32_t word = w[e >> 1];
        return bf16_bits_to_f32((e & 1) ? (word >> 16) : (word & 0xffffu));
    }
};

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool valid)
{
    const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
    const int bytes = valid ? 16 : 0;  // 0: the 16 bytes are zero-filled, nothing is read
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

__host__ __device__ constexpr size_t round16(size_t b) { return (b + 15) / 16 * 16; }

template <typename TS, int G, int K, int MG, int T, int D, int WC>
struct RegTile {
    static constexpr int kThreads = 256;
    static constexpr int kRC = 16;                        // reduction indices per chunk
    static constexpr int kVec = Elem<TS>::kVec;
    static constexpr int kWN = 8 / WC;                    // column-warps
    static constexpr int kNTC = kWN * 32 * T;             // columns per CTA
    static constexpr int kNGR = WC * MG;                  // groups per CTA
    static constexpr int kSlots = kRC * K;                // slots of one group in a chunk
    static constexpr bool kExpand = D == 0;               // branch-free: G decompressed weights
    static constexpr int kDisp = kExpand ? 0 : K / D;     // jumps per (group, r)
    static constexpr int kWords = D > 1 ? K / D : (K + 3) / 4;
    static constexpr int kRecVec =
        kExpand ? G / 4 : static_cast<int>(round16(4 * K + 4 * kWords) / 16);
    static constexpr int kXPitch = kRC + 16 / static_cast<int>(sizeof(TS));
    static_assert(WC == 4 || WC == 8, "4 or 8 channel-warps");
    static_assert(D == 0 || D == 1 || (D == 2 && K % 2 == 0), "expand, or one or two slots per jump");
    static_assert(D != 0 || G % 4 == 0, "expanded records are whole 16-byte units");
    static_assert(T % 4 == 0, "T must be a multiple of 4");
    static_assert(kRC % kVec == 0, "a chunk must hold whole 16-byte vectors");
    static_assert((kSlots * static_cast<int>(sizeof(TS))) % 16 == 0, "value runs must be 16-byte multiples");
    static_assert(kSlots % 16 == 0, "index runs must be 16-byte multiples");
    static_assert((MG * G) % 4 == 0, "output rows are stored as float4");

    // shared-memory layout (byte offsets; every part 16-byte aligned)
    static constexpr size_t kXraw = 0;
    static constexpr size_t kXs = kXraw + round16(2ull * kNTC * kXPitch * sizeof(TS));
    static constexpr size_t kVraw = kXs + round16(2ull * kRC * kNTC * sizeof(float));
    static constexpr size_t kIraw = kVraw + round16(2ull * kNGR * kSlots * sizeof(TS));
    static constexpr size_t kRec = kIraw + round16(2ull * kNGR * kSlots);
    static constexpr size_t kSites = kRec + round16(2ull * kNGR * kRC * kRecVec * 16);
    static constexpr size_t kTotal = kSites + round16(static_cast<size_t>(kNTC) * sizeof(int4));
};

__device__ __forceinline__ uint32_t word_of(const uint4 &u, int k)
{
    return k == 0 ? u.x : k == 1 ? u.y : k == 2 ? u.z : u.w;
}

// ---------------------------------------------------------------------------
// the kernel: persistent over tiles (tile = channel tile fastest, so the CTAs
// running at the same time share column tiles and X is reused through L2)
// ---------------------------------------------------------------------------
// CTAs per SM the kernel is compiled for: two when the accumulator tile is at
// most 64 fp32 registers per lane (16 resident warps hide the shared-load and
// barrier latencies), else one
template <int MG, int G, int T>
constexpr int regtile_min_blocks() { return MG * G * T <= 64 ? 2 : 1; }

template <typename TS, int G, int K, int MG, int T, int D, int WC>
__global__ void __launch_bounds__(256, regtile_min_blocks<MG, G, T>())
    regtile_kernel(FwdParams p, int64_t n_ct, int64_t n_tiles)
{
    using RT = RegTile<TS, G, K, MG, T, D, WC>;
    constexpr int RC = RT::kRC;
    constexpr int VEC = RT::kVec;
    constexpr int NTC = RT::kNTC;
    constexpr int NGR = RT::kNGR;
    constexpr int SLOTS = RT::kSlots;
    constexpr int XP = RT::kXPitch;
    constexpr int RV = RT::kRecVec;
    constexpr int H = T / 2;
    extern __shared__ __align__(16) unsigned char smem[];
    TS *xraw = reinterpret_cast<TS *>(smem + RT::kXraw);
    float *xs = reinterpret_cast<float *>(smem + RT::kXs);
    TS *vraw = reinterpret_cast<TS *>(smem + RT::kVraw);
    uint8_t *iraw = smem + RT::kIraw;
    uint4 *rec = reinterpret_cast<uint4 *>(smem + RT::kRec);
    int4 *sites = reinterpret_cast<int4 *>(smem + RT::kSites);

    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int wcw = warp % WC;  // channel-warp index
    const int wnw = warp / WC;  // column-warp index
    const int64_t total_groups = p.Cout / G;
    const int nchunks = static_cast<int>((p.R + RC - 1) / RC);
    const TS *X = static_cast<const TS *>(p.X);
    const TS *V = static_cast<const TS *>(p.values);

    for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int64_t ct = tile % n_ct;
        const int64_t n0 = (tile / n_ct) * NTC;
        const int64_t g0 = ct * NGR;  // first group of the CTA

        // column sites: {img lo, img hi (-1: column past N), hb, wb}
        for (int c = tid; c < NTC; c += RT::kThreads) {
            const int64_t n = n0 + c;
            int4 s = make_int4(0, -1, 0, 0);
            if (n < p.N) {
                const ColumnSite cs = column_site(p, n);
                s = make_int4(static_cast<int>(cs.img & 0xffffffffll), static_cast<int>(cs.img >> 32), cs.hb,
                              cs.wb);
            }
            sites[c] = s;
        }
        __syncthreads();

        auto issue_chunk = [&](int chunk) {
            const int buf = chunk & 1;
            const int64_t r0 = static_cast<int64_t>(chunk) * RC;
            TS *xr = xraw + buf * (NTC * XP);
#pragma unroll
            for (int it = 0; it < (NTC * (RC / VEC) + RT::kThreads - 1) / RT::kThreads; ++it) {
                const int v = it * RT::kThreads + tid;
                if (v < NTC * (RC / VEC)) {
                    const int col = v % NTC;
                    const int rv = v / NTC;
                    const int64_t r = r0 + rv * VEC;
                    const int4 s = sites[col];
                    bool ok = (s.y >= 0) && (r < p.R);
                    const TS *src = X;
                    if (ok) {
                        const int64_t img = (static_cast<int64_t>(s.y) << 32) | static_cast<uint32_t>(s.x);
                        if (!p.is_conv) {
                            src = X + img + r;
                        } else {
                            const int64_t tap = r / p.Cin;
                            const int64_t ci = r - tap * p.Cin;
                            const int kh = static_cast<int>(tap / p.KW);
                            const int kw = static_cast<int>(tap - static_cast<int64_t>(kh) * p.KW);
                            const int h = s.z + kh, w = s.w + kw;
                            ok = (h >= 0) && (h < p.H) && (w >= 0) && (w < p.W);
                            if (ok) src = X + img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
                        }
                    }
                    cp_async16(xr + col * XP + rv * VEC, src, ok);
                }
            }
            TS *vr = vraw + buf * (NGR * SLOTS);
            uint8_t *ir = iraw + buf * (NGR * SLOTS);
            constexpr int EPV = 16 / static_cast<int>(sizeof(TS));  // values per 16 bytes
            constexpr int VPG = SLOTS / EPV;                          // value vectors per group
            constexpr int IPG = SLOTS / 16;                           // index vectors per group
            for (int v = tid; v < NGR * (VPG + IPG); v += RT::kThreads) {
                const int gl = v / (VPG + IPG);
                const int part = v % (VPG + IPG);
                const int64_t gg = g0 + gl;
                if (part < VPG) {
                    const int e0 = part * EPV;
                    const bool ok = gg < total_groups && r0 + e0 / K < p.R;
                    cp_async16(vr + gl * SLOTS + e0, ok ? V + (gg * p.R + r0) * K + e0 : V, ok);
                } else {
                    const int e0 = (part - VPG) * 16;
                    const bool ok = gg < total_groups && r0 + e0 / K < p.R;
                    cp_async16(ir + gl * SLOTS + e0, ok ? p.idx + (gg * p.R + r0) * K + e0 : p.idx, ok);
                }
            }
            cp_async_commit();
        };

        auto transform_chunk = [&](int chunk) {
            const int buf = chunk & 1;
            const int64_t r0 = static_cast<int64_t>(chunk) * RC;
            const TS *xr = xraw + buf * (NTC * XP);
            float *xo = xs + buf * (RC * NTC);
#pragma unroll
            for (int it = 0; it < (NTC * (RC / VEC) + RT::kThreads - 1) / RT::kThreads; ++it) {
                const int v = it * RT::kThreads + tid;
                if (v < NTC * (RC / VEC)) {
                    const int col = v % NTC;
                    const int rv = v / NTC;
                    const uint4 w4 = *reinterpret_cast<const uint4 *>(xr + col * XP + rv * VEC);
                    const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                    for (int e = 0; e < VEC; ++e) xo[(rv * VEC + e) * NTC + col] = Elem<TS>::widen(w, e);
                }
            }
            const TS *vr = vraw + buf * (NGR * SLOTS);
            const uint8_t *ir = iraw + buf * (NGR * SLOTS);
            uint4 *ro = rec + buf * (NGR * RC * RV);
            if constexpr (RT::kExpand) {
                // record = the G weights of (group, r) with the pruned ones zero;
                // the thread owns the record, so the zero fill and the adds need no sync
                for (int item = tid; item < NGR * RC; item += RT::kThreads) {
                    const int gl = item / RC;
                    const int r = item % RC;
                    const bool live = (g0 + gl < total_groups) && (r0 + r < p.R);
                    // every write of the record goes through float (one type for the
                    // zero fill and the adds, so no aliasing reordering between them)
                    float *w = reinterpret_cast<float *>(ro + (gl * RC + r) * RV);
#pragma unroll
                    for (int q = 0; q < RV; ++q)
                        reinterpret_cast<float4 *>(w)[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                    if (!live) continue;
#pragma unroll
                    for (int s = 0; s < K; ++s) {
                        const float v = Elem<TS>::to_f32(vr[gl * SLOTS + r * K + s]);
                        const int i = ir[gl * SLOTS + r * K + s];
                        if (i >= G) {
                            report(p.status, CCI_ERR_INDEX);
                            continue;
                        }
                        w[i] += v;  // a repeated index adds both values
                    }
                }
                return;
            }
            for (int item = tid; item < NGR * RC; item += RT::kThreads) {
                const int gl = item / RC;
                const int r = item % RC;
                const bool live = (g0 + gl < total_groups) && (r0 + r < p.R);
                uint32_t words[RV * 4];
#pragma unroll
                for (int k = 0; k < RV * 4; ++k) words[k] = 0;
                int idxs[K];
#pragma unroll
                for (int s = 0; s < K; ++s) {
                    float v = 0.0f;
                    int i = s % G;  // padding: value 0 on an ascending index set
                    if (live) {
                        v = Elem<TS>::to_f32(vr[gl * SLOTS + r * K + s]);
                        i = ir[gl * SLOTS + r * K + s];
                        if (i >= G) {
                            report(p.status, CCI_ERR_INDEX);
                            v = 0.0f;
                            i = 0;
                        }
                    }
                    words[s] = __float_as_uint(v);
                    idxs[s] = i;
                }
                if constexpr (D == 1) {
#pragma unroll
                    for (int s = 0; s < K; ++s) words[K + s / 4] |= static_cast<uint32_t>(idxs[s]) << (8 * (s % 4));
                } else {
#pragma unroll
                    for (int d = 0; d < K / 2; ++d) {
                        const int i0 = idxs[2 * d], i1 = idxs[2 * d + 1];
                        const uint32_t code = (i0 < i1) ? static_cast<uint32_t>(i0 + i1 * (i1 - 1) / 2)
                                                        : static_cast<uint32_t>(G * (G - 1) / 2);
                        words[K + d] = code | (static_cast<uint32_t>(i0) << 8) | (static_cast<uint32_t>(i1) << 16);
                    }
                }
                uint4 *dst = ro + (gl * RC + r) * RV;
#pragma unroll
                for (int q = 0; q < RV; ++q)
                    dst[q] = make_uint4(words[4 * q], words[4 * q + 1], words[4 * q + 2], words[4 * q + 3]);
            }
        };

        unsigned long long acc[MG][G][H];
#pragma unroll
        for (int g = 0; g < MG; ++g)
#pragma unroll
            for (int i = 0; i < G; ++i)
#pragma unroll
                for (int t = 0; t < H; ++t) acc[g][i][t] = 0ull;

        // Buffer safety (b = chunk parity):
        //  * issue(c+1) writes raw[b'] last read by transform(c-1): separated by the
        //    barriers of iteration c-1;
        //  * transform(c+1) writes xs/rec[b'] last read by compute(c-1): separated by
        //    the barrier before compute(c);
        //  * compute(c) reads xs/rec[b] written by transform(c): barrier before compute.
        issue_chunk(0);
        cp_async_wait_all();
        __syncthreads();
        transform_chunk(0);
        for (int c = 0; c < nchunks; ++c) {
            if (c + 1 < nchunks) issue_chunk(c + 1);
            __syncthreads();
            const int buf = c & 1;
            const float *xw = xs + buf * (RC * NTC) + wnw * (32 * T) + lane * 4;
            const uint4 *rw = rec + buf * (NGR * RC * RV) + wcw * MG * RC * RV;

            if constexpr (RT::kExpand) {
                // straight-line code: unrolled so the compiler schedules the shared
                // loads of later reduction indices under the FMAs of earlier ones
#pragma unroll 4
                for (int r = 0; r < RC; ++r) {
                    unsigned long long xx[H];
#pragma unroll
                    for (int q = 0; q < T / 4; ++q) {
                        const ulonglong2 u = *reinterpret_cast<const ulonglong2 *>(xw + r * NTC + q * 128);
                        xx[2 * q] = u.x;
                        xx[2 * q + 1] = u.y;
                    }
#pragma unroll
                    for (int g = 0; g < MG; ++g) {
#pragma unroll
                        for (int q = 0; q < RV; ++q) {
                            const float4 w4 = reinterpret_cast<const float4 *>(rw)[(g * RC + r) * RV + q];
                            const float w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const unsigned long long ww = pack2(w[e], w[e]);
#pragma unroll
                                for (int t = 0; t < H; ++t) ffma2(acc[g][4 * q + e][t], xx[t], ww);
                            }
                        }
                    }
                }
            } else {
            unsigned long long xx[H];
            uint4 rc[MG][RV];
            auto load_r = [&](int r, unsigned long long (&xo)[H], uint4 (&ro)[MG][RV]) {
#pragma unroll
                for (int q = 0; q < T / 4; ++q) {
                    const ulonglong2 u = *reinterpret_cast<const ulonglong2 *>(xw + r * NTC + q * 128);
                    xo[2 * q] = u.x;
                    xo[2 * q + 1] = u.y;
                }
#pragma unroll
                for (int g = 0; g < MG; ++g)
#pragma unroll
                    for (int q = 0; q < RV; ++q) ro[g][q] = rw[(g * RC + r) * RV + q];
            };
            load_r(0, xx, rc);
#pragma unroll 1
            for (int r = 0; r < RC; ++r) {
                unsigned long long xn[H];
                uint4 rn[MG][RV];
                load_r(r + 1 < RC ? r + 1 : r, xn, rn);  // prefetch the next reduction index
                {
#pragma unroll
                for (int g = 0; g < MG; ++g) {
#pragma unroll
                    for (int d = 0; d < RT::kDisp; ++d) {
                        constexpr int DD = D > 0 ? D : 1;
                        unsigned long long vv[DD];
#pragma unroll
                        for (int s = 0; s < DD; ++s) {
                            const float v = __uint_as_float(word_of(rc[g][(d * DD + s) / 4], (d * DD + s) % 4));
                            vv[s] = pack2(v, v);
                        }
                        uint32_t word;
                        if constexpr (DD == 1) {
                            word = (word_of(rc[g][(K + d / 4) / 4], (K + d / 4) % 4) >> (8 * (d % 4))) & 0xffu;
                        } else {
                            word = word_of(rc[g][(K + d) / 4], (K + d) % 4);
                        }
                        Dispatch<G, (D > 0 ? D : 1), T>::run(acc[g], xx, vv, word);
                    }
                }
                }
#pragma unroll
                for (int t = 0; t < H; ++t) xx[t] = xn[t];
#pragma unroll
                for (int g = 0; g < MG; ++g)
#pragma unroll
                    for (int q = 0; q < RV; ++q) rc[g][q] = rn[g][q];
            }
            }  // jump-dispatch path
            if (c + 1 < nchunks) {
                cp_async_wait_all();
                __syncthreads();
                transform_chunk(c + 1);
            }
        }

        // epilogue: Y[n][c0 .. c0 + MG*G) for this lane's T columns
        const int64_t gfirst = g0 + wcw * MG;
#pragma unroll
        for (int t2 = 0; t2 < H; ++t2) {
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int col = wnw * (32 * T) + (t2 >> 1) * 128 + lane * 4 + (t2 & 1) * 2 + e;
                const int64_t n = n0 + col;
                if (n >= p.N) continue;
                float *yrow = p.Y + n * p.Cout;
#pragma unroll
                for (int g = 0; g < MG; ++g) {
                    if (gfirst + g >= total_groups) continue;
                    float4 *yg = reinterpret_cast<float4 *>(yrow + (gfirst + g) * G);
#pragma unroll
                    for (int i4 = 0; i4 < G / 4; ++i4) {
                        float4 o;
                        o.x = e ? hi_of(acc[g][4 * i4 + 0][t2]) : lo_of(acc[g][4 * i4 + 0][t2]);
                        o.y = e ? hi_of(acc[g][4 * i4 + 1][t2]) : lo_of(acc[g][4 * i4 + 1][t2]);
                        o.z = e ? hi_of(acc[g][4 * i4 + 2][t2]) : lo_of(acc[g][4 * i4 + 2][t2]);
                        o.w = e ? hi_of(acc[g][4 * i4 + 3][t2]) : lo_of(acc[g][4 * i4 + 3][t2]);
                        __stcs(yg + i4, o);
                    }
                }
            }
        }
        __syncthreads();  // shared memory is reused by the next tile
    }
}

}  // namespace cci
