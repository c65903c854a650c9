// cci_basic.cu -- the pack kernel, the targeted-dropout mask, the allocation
// statistics of packing, the generic product kernel and the FMA probe.
#include <type_traits>

#include "cci_kernels.h"

namespace cci {

// ---------------------------------------------------------------------------
// pack: one thread per (group gi, input feature r); this general form takes
// any G <= 256 and re-reads the column from cache while ranking.  Sec. 3.1 / Sec. 5.1:
// the K weights of largest |w| in W[gi*G .. gi*G+G)[r] survive, ties to the
// lower index, and are written in increasing index.  |w| is compared on the
// storage bits with the sign cleared (an order-preserving integer compare for
// every non-NaN value; NaN bit patterns rank above +inf and are reported).
// ---------------------------------------------------------------------------
template <typename TB>  // uint32_t for fp32, uint16_t for bf16 (raw bits)
__global__ void pack_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int G, int K,
                            TB *__restrict__ values, uint8_t *__restrict__ idx, uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    const int64_t total = (Cout / G) * R;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gi = t / R;
        const int64_t r = t - gi * R;
        const TB *col = W + gi * G * R + r;
        bool nan = false;
        int s = 0;
        for (int j = 0; j < G && s < K; ++j) {
            const TB wj = col[static_cast<int64_t>(j) * R];
            const uint32_t a = static_cast<uint32_t>(wj) & kAbs;
            nan |= a > kInf;
            int rank = 0;  // number of entries ranked ahead of j
            for (int j2 = 0; j2 < G && rank < K; ++j2) {
                const uint32_t b = static_cast<uint32_t>(col[static_cast<int64_t>(j2) * R]) & kAbs;
                rank += (b > a) || (b == a && j2 < j);
            }
            if (rank < K) {
                values[t * K + s] = wj;
                idx[t * K + s] = static_cast<uint8_t>(j);
                ++s;
            }
        }
        // entries after the K-th survivor were not scanned; check them for NaN too
        for (int j = 0; j < G; ++j)
            nan |= (static_cast<uint32_t>(col[static_cast<int64_t>(j) * R]) & kAbs) > kInf;
        if (nan) report(status, CCI_ERR_VALUE);
    }
}

// Register form for the group sizes of every workload (G <= 32, a power of
// two): the G entries of the column are loaded once, coalesced across the
// warp (consecutive threads take consecutive r), and ranked in registers.
template <typename TB, int GT>
__global__ void __launch_bounds__(128) pack_reg_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int K,
                                                       TB *__restrict__ values, uint8_t *__restrict__ idx,
                                                       uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    const int64_t total = (Cout / GT) * R;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gi = t / R;
        const int64_t r = t - gi * R;
        const TB *col = W + gi * GT * R + r;
        TB w[GT];
        uint32_t a[GT];
#pragma unroll
        for (int j = 0; j < GT; ++j) {
            w[j] = __ldg(col + static_cast<int64_t>(j) * R);
            a[j] = static_cast<uint32_t>(w[j]) & kAbs;
        }
        bool nan = false;
        int s = 0;
#pragma unroll
        for (int j = 0; j < GT; ++j) {
            nan |= a[j] > kInf;
            int rank = 0;  // entries ranked ahead of j: larger |w|, or equal |w| at a lower index
#pragma unroll
            for (int j2 = 0; j2 < GT; ++j2)
                rank += j2 < j ? (a[j2] >= a[j]) : (a[j2] > a[j]);
            if (rank < K) {
                values[t * K + s] = w[j];
                idx[t * K + s] = static_cast<uint8_t>(j);
                ++s;
            }
        }
        if (nan) report(status, CCI_ERR_VALUE);
    }
}

// Vector form of the register kernel: each thread ranks four consecutive
// columns r0 .. r0 + 3 of one group, its G rows loaded as one 8-byte (bf16) or
// 16-byte (fp32) vector each; the group is the block's y index, so no thread
// divides.  The K kept (value, index) pairs of a column are gathered in 64-bit
// registers (slot s at bit s * element width) and the four columns' outputs,
// contiguous in the packed arrays, are written with 16-byte stores.  Needs
// R % 4 == 0, W, values and idx 16-byte aligned, Cout / G <= 65535 and
// K * element bits <= 64 with 4 K elements a multiple of 16 bytes (bf16: K in
// {2, 4}; fp32: K in {1, 2}).
template <typename TB, int GT, int KT>
__global__ void __launch_bounds__(128) pack_vec_kernel(const TB *__restrict__ W, int64_t R, TB *__restrict__ values,
                                                       uint8_t *__restrict__ idx, uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    constexpr int kBits = 8 * sizeof(TB);
    const int64_t gi = blockIdx.y;
    const int64_t r0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) * 4;
    if (r0 >= R) return;
    const TB *col = W + gi * GT * R + r0;
    TB w[GT][4];
#pragma unroll
    for (int j = 0; j < GT; ++j) {
        if constexpr (sizeof(TB) == 4) {
            const uint4 x = __ldg(reinterpret_cast<const uint4 *>(col + static_cast<int64_t>(j) * R));
            w[j][0] = x.x;
            w[j][1] = x.y;
            w[j][2] = x.z;
            w[j][3] = x.w;
        } else {
            const uint2 x = __ldg(reinterpret_cast<const uint2 *>(col + static_cast<int64_t>(j) * R));
            w[j][0] = static_cast<TB>(x.x);
            w[j][1] = static_cast<TB>(x.x >> 16);
            w[j][2] = static_cast<TB>(x.y);
            w[j][3] = static_cast<TB>(x.y >> 16);
        }
    }
    bool nan = false;
    uint64_t ov[4], oi[4];  // per column: kept values and indices, slot s at s * width
    // ranking keys: the magnitude bits, then the inverted index, then the sign:
    // keys are distinct, a larger key is a larger |w| or an equal |w| at a lower
    // index (the tie rule; the sign ranks nothing), and a key gives back its entry
    // (value = sign and magnitude, index = 255 - the index field).  The K kept
    // entries are the K largest keys, kept sorted while the G keys pass once
    // (insertion: slot s takes the larger of itself and the smaller of slot s - 1
    // and the key), then put in increasing index.  A NaN magnitude outranks every
    // other key, so the column holds a NaN exactly when its largest key does.
    using Key = typename std::conditional<sizeof(TB) == 4, uint64_t, uint32_t>::type;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        Key sel[KT];
#pragma unroll
        for (int k = 0; k < KT; ++k) sel[k] = 0;  // every key is above 0 (its index field is not 0)
#pragma unroll
        for (int j = 0; j < GT; ++j) {
            const uint32_t b = static_cast<uint32_t>(w[j][v]);
            // the fields do not overlap: a multiply-add builds the key (FMA pipe)
            const Key key = static_cast<Key>(b & kAbs) * 512u + static_cast<Key>(((255 - j) << 1) + (b >> (kBits - 1)));
#pragma unroll
            for (int k = KT - 1; k > 0; --k) {
                const Key lo = sel[k - 1] < key ? sel[k - 1] : key;
                sel[k] = sel[k] > lo ? sel[k] : lo;
            }
            sel[0] = sel[0] > key ? sel[0] : key;
        }
        nan |= (sel[0] >> 9) > kInf;
        // increasing index = decreasing inverted-index field
#pragma unroll
        for (int a = 0; a < KT; ++a)
#pragma unroll
            for (int b = 0; b + 1 < KT - a; ++b) {
                const Key x = sel[b], y = sel[b + 1];
                const bool swap = ((x >> 1) & 255) < ((y >> 1) & 255);
                sel[b] = swap ? y : x;
                sel[b + 1] = swap ? x : y;
            }
        uint64_t vv = 0, ii = 0;
#pragma unroll
        for (int k = 0; k < KT; ++k) {
            const uint64_t value = static_cast<uint64_t>((sel[k] >> 9) | (static_cast<Key>(sel[k] & 1) << (kBits - 1)));
            vv |= value << (k * kBits);
            ii |= static_cast<uint64_t>(255 - ((sel[k] >> 1) & 255)) << (8 * k);
        }
        ov[v] = vv;
        oi[v] = ii;
    }
    // values of the four columns: 4 K elements from (gi * R + r0) * K on
    const int64_t t0 = (gi * R + r0) * KT;
    constexpr int kVB = KT * kBits;  // bits of one column's values (32 or 64)
    uint4 *pv = reinterpret_cast<uint4 *>(values + t0);
    if constexpr (kVB == 32) {
        pv[0] = make_uint4(static_cast<uint32_t>(ov[0]), static_cast<uint32_t>(ov[1]), static_cast<uint32_t>(ov[2]),
                           static_cast<uint32_t>(ov[3]));
    } else {
        pv[0] = make_uint4(static_cast<uint32_t>(ov[0]), static_cast<uint32_t>(ov[0] >> 32),
                           static_cast<uint32_t>(ov[1]), static_cast<uint32_t>(ov[1] >> 32));
        pv[1] = make_uint4(static_cast<uint32_t>(ov[2]), static_cast<uint32_t>(ov[2] >> 32),
                           static_cast<uint32_t>(ov[3]), static_cast<uint32_t>(ov[3] >> 32));
    }
    // indices: 4 K bytes
    if constexpr (KT == 1) {
        *reinterpret_cast<uint32_t *>(idx + t0) = static_cast<uint32_t>(oi[0] | (oi[1] << 8) | (oi[2] << 16) | (oi[3] << 24));
    } else if constexpr (KT == 2) {
        *reinterpret_cast<uint2 *>(idx + t0) = make_uint2(static_cast<uint32_t>(oi[0] | (oi[1] << 16)),
                                                          static_cast<uint32_t>(oi[2] | (oi[3] << 16)));
    } else {
        *reinterpret_cast<uint4 *>(idx + t0) = make_uint4(static_cast<uint32_t>(oi[0]), static_cast<uint32_t>(oi[1]),
                                                          static_cast<uint32_t>(oi[2]), static_cast<uint32_t>(oi[3]));
    }
    if (nan) report(status, CCI_ERR_VALUE);
    // a programmatic dependent (the decompression of the product that follows)
    // may be scheduled once every block got here; it waits for this grid's
    // completion before reading the packed arrays
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename TB>
cudaError_t launch_pack_t(const TB *W, int64_t Cout, int64_t R, int G, int K, TB *values, uint8_t *idx,
                          uint32_t *status, cudaStream_t stream)
{
    const int64_t total = (Cout / G) * R;
    const bool reg = G == 2 || G == 4 || G == 8 || G == 16 || G == 32;
    const bool vec_k = sizeof(TB) == 2 ? (K == 2 || K == 4) : (K == 1 || K == 2);
    const bool vec_g = (G == 4 && K <= 2) || (G == 8 && K <= 4) || (G == 16 && K <= 4) || (G == 32 && K <= 4);
    if (vec_k && vec_g && R % 4 == 0 && Cout / G <= 65535 && reinterpret_cast<uintptr_t>(W) % 16 == 0 &&
        reinterpret_cast<uintptr_t>(values) % 16 == 0 && reinterpret_cast<uintptr_t>(idx) % 16 == 0 &&
        (R / 4 + 127) / 128 <= 0x7fffffff) {
        const dim3 grid(static_cast<unsigned>((R / 4 + 127) / 128), static_cast<unsigned>(Cout / G));
#define CCI_PACK_VEC(g, k)                                                                          \
    if (G == g && K == k) {                                                                         \
        pack_vec_kernel<TB, g, k><<<grid, 128, 0, stream>>>(W, R, values, idx, status);            \
        return cudaGetLastError();                                                                  \
    }
        if constexpr (sizeof(TB) == 2) {
            CCI_PACK_VEC(4, 2) CCI_PACK_VEC(8, 2) CCI_PACK_VEC(8, 4) CCI_PACK_VEC(16, 2) CCI_PACK_VEC(16, 4)
            CCI_PACK_VEC(32, 2) CCI_PACK_VEC(32, 4)
        } else {
            CCI_PACK_VEC(4, 1) CCI_PACK_VEC(4, 2) CCI_PACK_VEC(8, 1) CCI_PACK_VEC(8, 2) CCI_PACK_VEC(16, 1)
            CCI_PACK_VEC(16, 2) CCI_PACK_VEC(32, 1) CCI_PACK_VEC(32, 2)
        }
#undef CCI_PACK_VEC
    }
    const int threads = reg ? 128 : 256;
    const int64_t blocks = (total + threads - 1) / threads;
    const int grid = static_cast<int>(blocks < 65536 * 16 ? blocks : 65536 * 16);
    switch (reg ? G : 0) {
        case 2: pack_reg_kernel<TB, 2><<<grid, threads, 0, stream>>>(W, Cout, R, K, values, idx, status); break;
        case 4: pack_reg_kernel<TB, 4><<<grid, threads, 0, stream>>>(W, Cout, R, K, values, idx, status); break;
        case 8: pack_reg_kernel<TB, 8><<<grid, threads, 0, stream>>>(W, Cout, R, K, values, idx, status); break;
        case 16: pack_reg_kernel<TB, 16><<<grid, threads, 0, stream>>>(W, Cout, R, K, values, idx, status); break;
        case 32: pack_reg_kernel<TB, 32><<<grid, threads, 0, stream>>>(W, Cout, R, K, values, idx, status); break;
        default: pack_kernel<TB><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, values, idx, status);
    }
    return cudaGetLastError();
}

cudaError_t launch_pack(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                        uint8_t *idx, uint32_t *status, cudaStream_t stream)
{
    if (dtype == CCI_F32)
        return launch_pack_t(static_cast<const uint32_t *>(W), Cout, R, G, K, static_cast<uint32_t *>(values), idx,
                             status, stream);
    return launch_pack_t(static_cast<const uint16_t *>(W), Cout, R, G, K, static_cast<uint16_t *>(values), idx,
                         status, stream);
}

// ---------------------------------------------------------------------------
// targeted dropout for CCI training (Sec. 5.1): per (group, r) the K weights of
// largest |w| (the ones pack keeps, same ranking and tie rule) are protected;
// every other weight is a pruning candidate and is zeroed for this pass when
// its uniform draw u < rate.  One thread per (group, r).
// ---------------------------------------------------------------------------
template <typename TB>
__global__ void td_mask_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int G, int K, float rate,
                               const float *__restrict__ u, TB *__restrict__ Wout, uint8_t *__restrict__ mask,
                               uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    const int64_t total = (Cout / G) * R;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gi = t / R;
        const int64_t r = t - gi * R;
        const TB *col = W + gi * G * R + r;
        bool nan = false;
        for (int j = 0; j < G; ++j) {
            const TB wj = col[static_cast<int64_t>(j) * R];
            const uint32_t a = static_cast<uint32_t>(wj) & kAbs;
            nan |= a > kInf;
            int rank = 0;  // number of entries ranked ahead of j
            for (int j2 = 0; j2 < G && rank < K; ++j2) {
                const uint32_t b = static_cast<uint32_t>(col[static_cast<int64_t>(j2) * R]) & kAbs;
                rank += (b > a) || (b == a && j2 < j);
            }
            const int64_t off = (gi * G + j) * R + r;
            const bool keep = rank < K || !(u[off] < rate);
            Wout[off] = keep ? wj : static_cast<TB>(0);
            if (mask) mask[off] = keep ? 1 : 0;
        }
        if (nan) report(status, CCI_ERR_VALUE);
    }
}

// Register form of the same step for G <= 32, a power of two: the column and
// its G uniform draws are loaded once (all loads in flight together) and the
// ranking runs in registers.
template <typename TB, int GT>
__global__ void __launch_bounds__(128) td_mask_reg_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int K,
                                                          float rate, const float *__restrict__ u,
                                                          TB *__restrict__ Wout, uint8_t *__restrict__ mask,
                                                          uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    const int64_t total = (Cout / GT) * R;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gi = t / R;
        const int64_t r = t - gi * R;
        const int64_t base = gi * GT * R + r;
        TB w[GT];
        float uj[GT];
        uint32_t a[GT];
#pragma unroll
        for (int j = 0; j < GT; ++j) {
            w[j] = __ldg(W + base + static_cast<int64_t>(j) * R);
            uj[j] = __ldg(u + base + static_cast<int64_t>(j) * R);
            a[j] = static_cast<uint32_t>(w[j]) & kAbs;
        }
        bool nan = false;
#pragma unroll
        for (int j = 0; j < GT; ++j) {
            nan |= a[j] > kInf;
            int rank = 0;  // entries ranked ahead of j: larger |w|, or equal |w| at a lower index
#pragma unroll
            for (int j2 = 0; j2 < GT; ++j2)
                rank += j2 < j ? (a[j2] >= a[j]) : (a[j2] > a[j]);
            const bool keep = rank < K || !(uj[j] < rate);
            const int64_t off = base + static_cast<int64_t>(j) * R;
            Wout[off] = keep ? w[j] : static_cast<TB>(0);
            if (mask) mask[off] = keep ? 1 : 0;
        }
        if (nan) report(status, CCI_ERR_VALUE);
    }
}

template <typename TB>
cudaError_t launch_td_mask_t(const TB *W, int64_t Cout, int64_t R, int G, int K, float rate, const float *u,
                             TB *Wout, uint8_t *mask, uint32_t *status, cudaStream_t stream)
{
    const int64_t total = (Cout / G) * R;
    const bool reg = G == 2 || G == 4 || G == 8 || G == 16 || G == 32;
    const int threads = reg ? 128 : 256;
    const int64_t blocks = (total + threads - 1) / threads;
    const int grid = static_cast<int>(blocks < 65536 * 16 ? blocks : 65536 * 16);
#define CCI_TD(GV) td_mask_reg_kernel<TB, GV><<<grid, threads, 0, stream>>>(W, Cout, R, K, rate, u, Wout, mask, status)
    switch (reg ? G : 0) {
        case 2: CCI_TD(2); break;
        case 4: CCI_TD(4); break;
        case 8: CCI_TD(8); break;
        case 16: CCI_TD(16); break;
        case 32: CCI_TD(32); break;
        default: td_mask_kernel<TB><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, rate, u, Wout, mask, status);
    }
#undef CCI_TD
    return cudaGetLastError();
}

cudaError_t launch_td_mask(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, float rate,
                           const float *u, void *Wout, uint8_t *mask, uint32_t *status, cudaStream_t stream)
{
    if (dtype == CCI_F32)
        return launch_td_mask_t(static_cast<const uint32_t *>(W), Cout, R, G, K, rate, u,
                                static_cast<uint32_t *>(Wout), mask, status, stream);
    return launch_td_mask_t(static_cast<const uint16_t *>(W), Cout, R, G, K, rate, u, static_cast<uint16_t *>(Wout),
                            mask, status, stream);
}

// ---------------------------------------------------------------------------
// allocation statistics of packing (Sec. 4, Eq. 1 measured on a weight matrix):
// per (group, r) the nonzero weights among the G and those beyond the K slots;
// one thread per (group, r), warp sums, one 64-bit atomic per warp and counter.
// A weight is nonzero when its magnitude bits are (so -0 is zero).
// ---------------------------------------------------------------------------
template <typename TB, int GT>  // GT = G known at compile time (all G loads in flight), or 0
__global__ void pack_stats_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int G_, int K,
                                  unsigned long long *counts)
{
    constexpr uint32_t kMag = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    const int G = GT ? GT : G_;
    const int64_t total = (Cout / G) * R;
    uint32_t nz_sum = 0, drop_sum = 0;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t gi = t / R, r = t - gi * R;
        const TB *w = W + gi * G * R + r;
        int nz = 0;
#pragma unroll
        for (int j = 0; j < G; ++j) nz += (static_cast<uint32_t>(__ldg(w + j * R)) & kMag) != 0;
        nz_sum += static_cast<uint32_t>(nz);
        drop_sum += static_cast<uint32_t>(nz > K ? nz - K : 0);
    }
    // block sum (warp shuffles, then the first warp over the warp sums), one
    // atomic per block and counter
    __shared__ unsigned long long part[2][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    nz_sum = __reduce_add_sync(0xffffffffu, nz_sum);
    drop_sum = __reduce_add_sync(0xffffffffu, drop_sum);
    if (lane == 0) {
        part[0][warp] = nz_sum;
        part[1][warp] = drop_sum;
    }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        unsigned long long a = lane < nw ? part[0][lane] : 0ull, b = lane < nw ? part[1][lane] : 0ull;
        for (int o = 16; o > 0; o >>= 1) {
            a += __shfl_down_sync(0xffffffffu, a, o);
            b += __shfl_down_sync(0xffffffffu, b, o);
        }
        if (lane == 0) {
            atomicAdd(counts, a);
            atomicAdd(counts + 1, b);
        }
    }
}

template <typename TB>
void launch_pack_stats_t(const TB *W, int64_t Cout, int64_t R, int G, int K, unsigned long long *counts,
                         cudaStream_t stream)
{
    const int64_t total = (Cout / G) * R;
    const int threads = 256;
    const int64_t blocks = (total + threads - 1) / threads;
    // at most 8 blocks per SM with grid-stride loops: few atomics; a thread's
    // sums stay far below 2^32 for any matrix that fits in memory
    const int grid = static_cast<int>(blocks < 152 * 8 ? blocks : 152 * 8);
    switch (G) {
        case 4: pack_stats_kernel<TB, 4><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, counts); break;
        case 8: pack_stats_kernel<TB, 8><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, counts); break;
        case 16: pack_stats_kernel<TB, 16><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, counts); break;
        case 32: pack_stats_kernel<TB, 32><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, counts); break;
        default: pack_stats_kernel<TB, 0><<<grid, threads, 0, stream>>>(W, Cout, R, G, K, counts);
    }
}

cudaError_t launch_pack_stats(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K,
                              unsigned long long *counts, cudaStream_t stream)
{
    if (dtype == CCI_F32)
        launch_pack_stats_t(static_cast<const uint32_t *>(W), Cout, R, G, K, counts, stream);
    else
        launch_pack_stats_t(static_cast<const uint16_t *>(W), Cout, R, G, K, counts, stream);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// generic product: any G <= 256, any K, any alignment.  A CTA of 128 threads
// owns one group and 128 columns; thread = column; the G accumulators of the
// column live in shared memory acc[G][128] (the thread's own column only).
// Contributions arrive in ascending r, then slot, each one fused multiply-add
// from +0 -- the same order as the register-tiled kernel.
// ---------------------------------------------------------------------------
template <typename TB>
__device__ __forceinline__ float load_elem(const TB *p, int64_t off);
template <>
__device__ __forceinline__ float load_elem<uint32_t>(const uint32_t *p, int64_t off)
{
    return __uint_as_float(__ldg(p + off));
}
template <>
__device__ __forceinline__ float load_elem<uint16_t>(const uint16_t *p, int64_t off)
{
    return bf16_bits_to_f32(__ldg(p + off));
}

template <typename TB>
__global__ void __launch_bounds__(128) generic_kernel(FwdParams p, int G, int K, int64_t n_col_tiles)
{
    extern __shared__ float acc[];  // [G][128]
    const int tid = threadIdx.x;
    const int64_t tile = blockIdx.x;
    const int64_t gi = tile / n_col_tiles;
    const int64_t n = (tile - gi * n_col_tiles) * 128 + tid;
    const bool col_ok = n < p.N;
    for (int i = 0; i < G; ++i) acc[i * 128 + tid] = 0.0f;
    ColumnSite site{0, 0, 0};
    if (col_ok) site = column_site(p, n);
    const TB *X = static_cast<const TB *>(p.X);
    const TB *V = static_cast<const TB *>(p.values) + gi * p.R * K;
    const uint8_t *I = p.idx + gi * p.R * K;
    bool bad = false;
    for (int64_t r = 0; r < p.R; ++r) {
        float x = 0.0f;
        if (col_ok) {
            const int64_t off = x_offset(p, site, r);
            if (off >= 0) x = load_elem<TB>(X, off);
        }
        for (int s = 0; s < K; ++s) {
            const int i = I[r * K + s];
            const float v = load_elem<TB>(V, r * K + s);
            if (i >= G) {
                bad = true;
                continue;
            }
            acc[i * 128 + tid] = fmaf(v, x, acc[i * 128 + tid]);
        }
    }
    if (bad && tid == 0) report(p.status, CCI_ERR_INDEX);
    if (col_ok) {
        float *y = p.Y + n * p.Cout + gi * G;
        for (int i = 0; i < G; ++i) y[i] = acc[i * 128 + tid];
    }
}

cudaError_t launch_generic(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream)
{
    const int64_t n_col_tiles = (p.N + 127) / 128;
    const int64_t tiles = n_col_tiles * (p.Cout / G);
    const size_t smem = static_cast<size_t>(G) * 128 * sizeof(float);
    static SmemAttrCache attr_f32, attr_bf16;
    const cudaError_t attr = dtype == CCI_F32 ? smem_attr_once(generic_kernel<uint32_t>, 256 * 128 * 4, attr_f32)
                                              : smem_attr_once(generic_kernel<uint16_t>, 256 * 128 * 4, attr_bf16);
    if (attr != cudaSuccess) return attr;
    if (tiles > 0x7fffffffll) return cudaErrorInvalidConfiguration;
    if (dtype == CCI_F32)
        generic_kernel<uint32_t><<<static_cast<unsigned>(tiles), 128, smem, stream>>>(p, G, K, n_col_tiles);
    else
        generic_kernel<uint16_t><<<static_cast<unsigned>(tiles), 128, smem, stream>>>(p, G, K, n_col_tiles);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// FMA probe: 16 independent packed-FMA chains per thread
// ---------------------------------------------------------------------------
__global__ void fma_probe_kernel(float *out, int iters)
{
    unsigned long long acc[16];
    const float seed = static_cast<float>(threadIdx.x) * 1e-3f;
#pragma unroll
    for (int k = 0; k < 16; ++k) acc[k] = pack2(seed + k, seed - k);
    const unsigned long long a = pack2(1.0e-3f, -1.0e-3f);
    const unsigned long long b = pack2(0.5f, 0.25f);
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int k = 0; k < 16; ++k) ffma2(acc[k], a, b);
    }
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < 16; ++k) s += lo_of(acc[k]) + hi_of(acc[k]);
    out[blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x] = s;
}

cudaError_t launch_fma_probe(float *out, int blocks, int threads, int iters, cudaStream_t stream)
{
    fma_probe_kernel<<<blocks, threads, 0, stream>>>(out, iters);
    return cudaGetLastError();
}

}  // namespace cci
