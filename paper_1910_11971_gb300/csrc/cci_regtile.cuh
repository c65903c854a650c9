// cci_regtile.cuh -- register-tiled CCI scatter kernel for sm_103a.
//
// Computes Alg. 2 of Sec. 3.2 (H(G*i + Idx, j) += Val * X(k, j), with a slot
// loop for K > 1) for a product or an implicit convolution.
//
// Work split (the group-boundary split of Sec. 3.2: a CTA owns whole groups):
//   * a CTA of 8 warps owns CH = WC*MG*G output channels (WC warps across
//     channels, each owning MG whole groups) and NTC = WN*32*T columns (WN = 8/WC
//     warps across columns);
//   * lane l of a warp owns T columns: 4-column runs at l*4 + q*128, q < T/4;
//   * every lane of a warp sees the same (value, index) pair at the same time
//     (the index depends on (group, r, slot), not on the column), so the index
//     choice of Alg. 2 is a warp-uniform branch, and the MG*G x T accumulator
//     block stays in registers ("load a whole group of elements of H onto
//     on-chip registers", Sec. 3.2);
//   * two columns share one packed FMA (fma.rn.f32x2), so a slot costs T/2 FMA
//     instructions per lane.
//
// Pipeline per chunk of RC reduction indices:
//   raw X tile [NTC][RC] and raw (value, index) runs are copied global->shared
//   with cp.async one chunk ahead (no registers held); the chunk is then
//   transposed to an fp32 [RC][NTC] tile (bf16 widened exactly) and the slots are
//   decoded into {v, v} pairs plus one dispatch code per (group, r): the colex
//   rank of the ascending index set among all K-subsets of [0, G) when there are
//   at most 128 subsets, else the raw indices.  A non-ascending or repeated index
//   set takes a per-slot path, so any index set is summed as Alg. 2 does.
//   Per output channel the contributions arrive in ascending r (then slot), each
//   one fused multiply-add, starting from +0.
#pragma once

#include "cci_common.cuh"

namespace cci {

__host__ __device__ constexpr int binom(int n, int k)
{
    if (k < 0 || k > n) return 0;
    long long r = 1;
    for (int i = 1; i <= k; ++i) r = r * (n - k + i) / i;
    return static_cast<int>(r);
}

// Element s (ascending) of the K-subset of [0, G) whose colex rank is c, where
// rank(i_0 < ... < i_{K-1}) = sum_s binom(i_s, s + 1).
__host__ __device__ constexpr int colex_element(int c, int K, int s)
{
    int out = 0;
    for (int t = K - 1; t >= 0; --t) {
        int i = t;
        while (binom(i + 1, t + 1) <= c) ++i;
        c -= binom(i, t + 1);
        if (t == s) out = i;
    }
    return out;
}

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

template <typename TS, int G, int K, int MG, int T>
struct RegTile {
    static constexpr int kThreads = 256;
    static constexpr int kWarps = 8;
    static constexpr int kRC = 16;          // reduction indices per chunk
    static constexpr int kVec = Elem<TS>::kVec;
    static constexpr int kNC = binom(G, K);
    static constexpr bool kCombo = kNC <= 128;
    static constexpr int kSlotsRC = kRC * K;  // slots of one group in a chunk
    static_assert(T % 4 == 0, "T must be a multiple of 4");
    static_assert(kRC % kVec == 0, "a chunk must hold whole 16-byte vectors");
    static_assert((kSlotsRC * static_cast<int>(sizeof(TS))) % 16 == 0, "value runs must be 16-byte multiples");
    static_assert(kSlotsRC % 16 == 0, "index runs must be 16-byte multiples");
    static_assert((MG * G) % 4 == 0, "output rows are stored as float4");

    // shared-memory layout (byte offsets; every part 16-byte aligned)
    struct Layout {
        int ntc;         // columns per CTA
        int ngroups;     // groups per CTA = WC * MG
        int xpitch;      // elements per raw X row (RC + 16 bytes of padding)
        size_t xraw, xs, vraw, iraw, vv, code, sidx, sites, total;
    };

    __host__ __device__ static Layout layout(int wc)
    {
        Layout L{};
        L.ntc = (kWarps / wc) * 32 * T;
        L.ngroups = wc * MG;
        L.xpitch = kRC + 16 / static_cast<int>(sizeof(TS));
        size_t off = 0;
        auto take = [&off](size_t bytes) {
            const size_t o = off;
            off += (bytes + 15) / 16 * 16;
            return o;
        };
        L.xraw = take(2ull * L.ntc * L.xpitch * sizeof(TS));
        L.xs = take(2ull * kRC * L.ntc * sizeof(float));
        L.vraw = take(2ull * L.ngroups * kSlotsRC * sizeof(TS));
        L.iraw = take(2ull * L.ngroups * kSlotsRC);
        L.vv = take(2ull * L.ngroups * kSlotsRC * sizeof(unsigned long long));
        L.code = take(2ull * L.ngroups * kRC);
        L.sidx = take(2ull * L.ngroups * kSlotsRC);
        L.sites = take(static_cast<size_t>(L.ntc) * sizeof(int4));
        L.total = off;
        return L;
    }
};

// ---------------------------------------------------------------------------
// slot application: acc[g][i][*] += x * v for a compile-time index i
// ---------------------------------------------------------------------------
template <int T, int G, int MG>
struct Acc {
    unsigned long long a[MG][G][T / 2];
};

template <int T, int G, int MG, int g, int i>
__device__ __forceinline__ void apply_slot(Acc<T, G, MG> &acc, const unsigned long long (&xx)[T / 2],
                                           unsigned long long v)
{
#pragma unroll
    for (int t = 0; t < T / 2; ++t) ffma2(acc.a[g][i][t], xx[t], v);
}

template <int T, int G, int MG, int g, int K, int c, int s = 0>
__device__ __forceinline__ void apply_combo(Acc<T, G, MG> &acc, const unsigned long long (&xx)[T / 2],
                                            const unsigned long long (&vv)[K])
{
    if constexpr (s < K) {
        constexpr int i = colex_element(c, K, s);
        apply_slot<T, G, MG, g, i>(acc, xx, vv[s]);
        apply_combo<T, G, MG, g, K, c, s + 1>(acc, xx, vv);
    }
}

#define CCI_CASE(c, BODY) \
    case (c):             \
        BODY(c);          \
        break;
#define CCI_CASES4(b, BODY) CCI_CASE(b, BODY) CCI_CASE(b + 1, BODY) CCI_CASE(b + 2, BODY) CCI_CASE(b + 3, BODY)
#define CCI_CASES16(b, BODY) \
    CCI_CASES4(b, BODY) CCI_CASES4(b + 4, BODY) CCI_CASES4(b + 8, BODY) CCI_CASES4(b + 12, BODY)
#define CCI_CASES64(b, BODY) \
    CCI_CASES16(b, BODY) CCI_CASES16(b + 16, BODY) CCI_CASES16(b + 32, BODY) CCI_CASES16(b + 48, BODY)
#define CCI_CASES128(b, BODY) CCI_CASES64(b, BODY) CCI_CASES64(b + 64, BODY)

// one slot with a run-time (warp-uniform) index: a G-way branch
template <int T, int G, int MG, int g>
__device__ __forceinline__ void apply_single(Acc<T, G, MG> &acc, const unsigned long long (&xx)[T / 2],
                                             unsigned long long v, int i)
{
#define CCI_SINGLE_BODY(c)                                         \
    if constexpr ((c) < G) {                                       \
        apply_slot<T, G, MG, g, ((c) < G ? (c) : 0)>(acc, xx, v); \
    }
    switch (i) {
        CCI_CASES128(0, CCI_SINGLE_BODY)
        default:
            break;
    }
#undef CCI_SINGLE_BODY
}

template <int T, int G, int MG, int g, int K>
__device__ __forceinline__ void apply_group(Acc<T, G, MG> &acc, const unsigned long long (&xx)[T / 2],
                                            const unsigned long long (&vv)[K], int code,
                                            const uint8_t *sidx)
{
    constexpr int NC = binom(G, K);
    if constexpr (NC <= 128) {
#define CCI_COMBO_BODY(c)                                               \
    if constexpr ((c) < NC) {                                           \
        apply_combo<T, G, MG, g, K, ((c) < NC ? (c) : 0)>(acc, xx, vv); \
    } else if constexpr ((c) == NC) {                                   \
        _Pragma("unroll") for (int s = 0; s < K; ++s)                   \
            apply_single<T, G, MG, g>(acc, xx, vv[s], sidx[s]);         \
    }
        switch (code) {
            CCI_CASES128(0, CCI_COMBO_BODY)
            CCI_CASE(128, CCI_COMBO_BODY)
            default:
                break;
        }
#undef CCI_COMBO_BODY
    } else {
#pragma unroll
        for (int s = 0; s < K; ++s) apply_single<T, G, MG, g>(acc, xx, vv[s], sidx[s]);
    }
}

// all MG groups of the warp at one reduction index r; the pointers are at
// (group 0, r) and advance by `gstride_*` per group
template <int T, int G, int MG, int K, int g = 0>
__device__ __forceinline__ void apply_all_groups(Acc<T, G, MG> &acc, const unsigned long long (&xx)[T / 2],
                                                 const unsigned long long *vv_r, const uint8_t *code_r,
                                                 const uint8_t *sidx_r, int gstride_code, int gstride_slot)
{
    if constexpr (g < MG) {
        unsigned long long vv[K];
#pragma unroll
        for (int s = 0; s < K; ++s) vv[s] = vv_r[g * gstride_slot + s];
        const int code = code_r[g * gstride_code];
        apply_group<T, G, MG, g, K>(acc, xx, vv, code, sidx_r + g * gstride_slot);
        apply_all_groups<T, G, MG, K, g + 1>(acc, xx, vv_r, code_r, sidx_r, gstride_code, gstride_slot);
    }
}

// ---------------------------------------------------------------------------
// the kernel: persistent over tiles (tile = channel tile fastest, so the CTAs
// running at the same time share column tiles and X is reused through L2)
// ---------------------------------------------------------------------------
template <typename TS, int G, int K, int MG, int T>
__global__ void __launch_bounds__(256, 1) regtile_kernel(FwdParams p, int wc, int64_t n_ct, int64_t n_tiles)
{
    using RT = RegTile<TS, G, K, MG, T>;
    constexpr int RC = RT::kRC;
    constexpr int VEC = RT::kVec;
    constexpr int SLOTS = RT::kSlotsRC;
    extern __shared__ __align__(16) unsigned char smem[];
    const auto L = RT::layout(wc);
    TS *xraw = reinterpret_cast<TS *>(smem + L.xraw);
    float *xs = reinterpret_cast<float *>(smem + L.xs);
    TS *vraw = reinterpret_cast<TS *>(smem + L.vraw);
    uint8_t *iraw = smem + L.iraw;
    unsigned long long *vvs = reinterpret_cast<unsigned long long *>(smem + L.vv);
    uint8_t *codes = smem + L.code;
    uint8_t *sidx = smem + L.sidx;
    int4 *sites = reinterpret_cast<int4 *>(smem + L.sites);

    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int wcw = warp % wc;  // channel-warp index
    const int wnw = warp / wc;  // column-warp index
    const int ntc = L.ntc;
    const int ngr = L.ngroups;
    const int xpitch = L.xpitch;
    const int64_t total_groups = p.Cout / G;
    const int nchunks = static_cast<int>((p.R + RC - 1) / RC);
    const TS *X = static_cast<const TS *>(p.X);
    const TS *V = static_cast<const TS *>(p.values);

    for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const int64_t ct = tile % n_ct;
        const int64_t n0 = (tile / n_ct) * ntc;
        const int64_t g0 = ct * ngr;  // first group of the CTA

        // column sites: {img lo, img hi (-1: column past N), hb, wb}
        for (int c = tid; c < ntc; c += RT::kThreads) {
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
            TS *xr = xraw + static_cast<size_t>(buf) * ntc * xpitch;
            const int nvec = ntc * (RC / VEC);
            for (int v = tid; v < nvec; v += RT::kThreads) {
                const int col = v % ntc;
                const int rv = v / ntc;
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
                cp_async16(xr + static_cast<size_t>(col) * xpitch + rv * VEC, src, ok);
            }
            TS *vr = vraw + static_cast<size_t>(buf) * ngr * SLOTS;
            uint8_t *ir = iraw + static_cast<size_t>(buf) * ngr * SLOTS;
            constexpr int VPG = SLOTS * static_cast<int>(sizeof(TS)) / 16;  // value vectors per group
            constexpr int EPV = 16 / static_cast<int>(sizeof(TS));          // values per vector
            constexpr int IPG = SLOTS / 16;                                 // index vectors per group
            const int nsv = ngr * (VPG + IPG);
            for (int v = tid; v < nsv; v += RT::kThreads) {
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
            const TS *xr = xraw + static_cast<size_t>(buf) * ntc * xpitch;
            float *xo = xs + static_cast<size_t>(buf) * RC * ntc;
            const int nvec = ntc * (RC / VEC);
            for (int v = tid; v < nvec; v += RT::kThreads) {
                const int col = v % ntc;
                const int rv = v / ntc;
                const uint4 w4 = *reinterpret_cast<const uint4 *>(xr + static_cast<size_t>(col) * xpitch + rv * VEC);
                const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    xo[static_cast<size_t>(rv * VEC + e) * ntc + col] = Elem<TS>::widen(w, e);
            }
            const TS *vr = vraw + static_cast<size_t>(buf) * ngr * SLOTS;
            const uint8_t *ir = iraw + static_cast<size_t>(buf) * ngr * SLOTS;
            unsigned long long *vo = vvs + static_cast<size_t>(buf) * ngr * SLOTS;
            uint8_t *co = codes + static_cast<size_t>(buf) * ngr * RC;
            uint8_t *so = sidx + static_cast<size_t>(buf) * ngr * SLOTS;
            const int nitems = ngr * RC;
            for (int it = tid; it < nitems; it += RT::kThreads) {
                const int gl = it / RC;
                const int r = it % RC;
                const bool live = (g0 + gl < total_groups) && (r0 + r < p.R);
                int code = 0, prev = -1;
                bool canon = true;
#pragma unroll
                for (int s = 0; s < K; ++s) {
                    float v = 0.0f;
                    int i = s;  // padding: value 0 on the index set {0..K-1}
                    if (live) {
                        v = Elem<TS>::to_f32(vr[gl * SLOTS + r * K + s]);
                        i = ir[gl * SLOTS + r * K + s];
                        if (i >= G) {
                            report(p.status, CCI_ERR_INDEX);
                            v = 0.0f;
                            i = 0;
                        }
                    }
                    canon = canon && (i > prev);
                    prev = i;
                    code += binom(i, s + 1);
                    vo[gl * SLOTS + r * K + s] = pack2(v, v);
                    so[gl * SLOTS + r * K + s] = static_cast<uint8_t>(i);
                }
                co[gl * RC + r] = static_cast<uint8_t>(canon ? code : RT::kNC);
            }
        };

        Acc<T, G, MG> acc;
#pragma unroll
        for (int g = 0; g < MG; ++g)
#pragma unroll
            for (int i = 0; i < G; ++i)
#pragma unroll
                for (int t = 0; t < T / 2; ++t) acc.a[g][i][t] = 0ull;

        // Buffer safety (b = chunk parity):
        //  * issue(c+1) writes raw[b'] last read by transform(c-1): separated by the
        //    barriers of iteration c-1;
        //  * transform(c+1) writes proc[b'] last read by compute(c-1): separated by
        //    the barrier before compute(c);
        //  * compute(c) reads proc[b] written by transform(c): barrier before compute.
        issue_chunk(0);
        cp_async_wait_all();
        __syncthreads();
        transform_chunk(0);
        for (int c = 0; c < nchunks; ++c) {
            if (c + 1 < nchunks) issue_chunk(c + 1);
            __syncthreads();
            const int buf = c & 1;
            const float *xo = xs + static_cast<size_t>(buf) * RC * ntc + wnw * (32 * T) + lane * 4;
            const int gw0 = wcw * MG;  // first CTA-local group of this warp
            const unsigned long long *vo = vvs + static_cast<size_t>(buf) * ngr * SLOTS + gw0 * SLOTS;
            const uint8_t *co = codes + static_cast<size_t>(buf) * ngr * RC + gw0 * RC;
            const uint8_t *so = sidx + static_cast<size_t>(buf) * ngr * SLOTS + gw0 * SLOTS;
#pragma unroll 1
            for (int r = 0; r < RC; ++r) {
                unsigned long long xx[T / 2];
#pragma unroll
                for (int q = 0; q < T / 4; ++q) {
                    const ulonglong2 u = *reinterpret_cast<const ulonglong2 *>(xo + r * ntc + q * 128);
                    xx[2 * q] = u.x;
                    xx[2 * q + 1] = u.y;
                }
                apply_all_groups<T, G, MG, K>(acc, xx, vo + r * K, co + r, so + r * K, RC, SLOTS);
            }
            if (c + 1 < nchunks) {
                cp_async_wait_all();
                __syncthreads();
                transform_chunk(c + 1);
            }
        }

        // epilogue: Y[n][c0 .. c0 + MG*G) for this lane's T columns
        const int64_t gfirst = g0 + wcw * MG;
#pragma unroll
        for (int t2 = 0; t2 < T / 2; ++t2) {
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
                        o.x = e ? hi_of(acc.a[g][4 * i4 + 0][t2]) : lo_of(acc.a[g][4 * i4 + 0][t2]);
                        o.y = e ? hi_of(acc.a[g][4 * i4 + 1][t2]) : lo_of(acc.a[g][4 * i4 + 1][t2]);
                        o.z = e ? hi_of(acc.a[g][4 * i4 + 2][t2]) : lo_of(acc.a[g][4 * i4 + 2][t2]);
                        o.w = e ? hi_of(acc.a[g][4 * i4 + 3][t2]) : lo_of(acc.a[g][4 * i4 + 3][t2]);
                        __stcs(yg + i4, o);
                    }
                }
            }
        }
        __syncthreads();  // shared memory is reused by the next tile
    }
}

}  // namespace cci
