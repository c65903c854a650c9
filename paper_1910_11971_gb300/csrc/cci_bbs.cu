// cci_bbs.cu -- balanced sparsity (Sec. 3.4), the format the paper compares CCI
// with: per output channel co, every group of G consecutive inputs
// r in [g*G, g*G + G) keeps K weights, stored as values[Cout][R/G][K] and
// idx[Cout][R/G][K] (offsets inside the group).  Its index selects an INPUT of
// the product (a gather), where CCI's selects an OUTPUT (a scatter).
//   bbs_pack_kernel        per (co, g): the K of largest |w|, ties to the lower
//                          index, in increasing index (CCI's selection rule)
//   bbs_decompress_kernel  per (co, g): the G dense weights of the group into the
//                          workspace of the tensor-core product (bf16, or the fp32
//                          operand planes), which then runs the CCI GEMM unchanged
//   bbs_gather_kernel      the product on CUDA cores (G dividing 32): X staged
//                          transposed in shared memory, each (value, index) pair
//                          reads one staged row (a warp-uniform address: no
//                          branch) into 4 FMAs per lane
#include "cci_kernels.h"

namespace cci {
namespace bbs {

template <typename TB>
__global__ void bbs_pack_kernel(const TB *__restrict__ W, int64_t Cout, int64_t R, int G, int K,
                                TB *__restrict__ values, uint8_t *__restrict__ idx, uint32_t *status)
{
    constexpr uint32_t kAbs = sizeof(TB) == 4 ? 0x7fffffffu : 0x7fffu;
    constexpr uint32_t kInf = sizeof(TB) == 4 ? 0x7f800000u : 0x7f80u;
    const int64_t ng = R / G;
    const int64_t total = Cout * ng;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const TB *grp = W + (t / ng) * R + (t % ng) * G;  // W[co][g*G ..]
        bool nan = false;
        int s = 0;
        for (int j = 0; j < G; ++j) {
            const TB wj = grp[j];
            const uint32_t a = static_cast<uint32_t>(wj) & kAbs;
            nan |= a > kInf;
            if (s == K) continue;
            int rank = 0;
            for (int j2 = 0; j2 < G && rank < K; ++j2) {
                const uint32_t b = static_cast<uint32_t>(grp[j2]) & kAbs;
                rank += (b > a) || (b == a && j2 < j);
            }
            if (rank < K) {
                values[t * K + s] = wj;
                idx[t * K + s] = static_cast<uint8_t>(j);
                ++s;
            }
        }
        if (nan) report(status, CCI_ERR_VALUE);
    }
}


// SPLIT: the two fp32 operand planes (store_w_split4) at w0 and w1; else the weights to w0.  Indices
// must be strictly increasing inside a group and < G (else CCI_ERR_INDEX).
// GC > 0: G == GC known at compile time, the group assembled in registers and
// written with 16-byte stores (G * element size a multiple of 16); GC == 0: any
// G, element stores.
template <typename TB, bool SPLIT, int GC>
__global__ void bbs_decompress_kernel(const TB *__restrict__ values, const uint8_t *__restrict__ idx, int64_t Cout,
                                      int64_t R, int G, int K, TB *__restrict__ w0, TB *__restrict__ w1,
                                      uint32_t *status)
{
    const int64_t ng = R / G;
    const int64_t total = Cout * ng;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t row = t / ng, c0 = (t % ng) * G;  // output channel, first index of the group
        const int64_t base = row * R + c0;
        int s = 0, prev = -1;
        bool bad = false;
        if constexpr (GC > 0) {
            TB g[GC];
            int ij = K > 0 ? idx[t * K] : -1;
#pragma unroll
            for (int j = 0; j < GC; ++j) {
                TB v = 0;
                if (s < K && ij == j) {
                    v = values[t * K + s];
                    bad |= ij <= prev;
                    prev = ij;
                    ++s;
                    ij = s < K ? idx[t * K + s] : -1;
                }
                g[j] = v;
            }
            bad |= s < K;  // an index >= G or out of order was never reached
            constexpr int kV = 16 / static_cast<int>(sizeof(TB));  // elements per 16-byte store
#pragma unroll
            for (int q = 0; q < GC / kV; ++q) {
                uint32_t h[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    if constexpr (sizeof(TB) == 4)
                        h[e] = static_cast<uint32_t>(g[q * kV + e]);
                    else
                        h[e] = static_cast<uint32_t>(g[q * kV + 2 * e]) |
                               (static_cast<uint32_t>(g[q * kV + 2 * e + 1]) << 16);
                }
                if constexpr (SPLIT)
                    store_w_split4(reinterpret_cast<uint32_t *>(w0), reinterpret_cast<uint16_t *>(w1), R, row,
                                   c0 + q * kV, h);
                else
                    reinterpret_cast<uint4 *>(w0 + base)[q] = make_uint4(h[0], h[1], h[2], h[3]);
            }
        } else {
            for (int j = 0; j < G; ++j) {
                TB v = 0;
                if (s < K) {
                    const int ij = idx[t * K + s];
                    bad |= ij >= G || ij <= prev;
                    if (ij == j) {
                        v = values[t * K + s];
                        prev = ij;
                        ++s;
                    }
                }
                if constexpr (SPLIT) {
                    store_w_split1(reinterpret_cast<uint32_t *>(w0), reinterpret_cast<uint16_t *>(w1), R, row, c0 + j,
                                   static_cast<uint32_t>(v));
                } else {
                    w0[base + j] = v;
                }
            }
            bad |= s < K;
        }
        if (bad) report(status, CCI_ERR_INDEX);
    }
}

template <typename TB>
__device__ __forceinline__ float to_f32(TB v)
{
    if constexpr (sizeof(TB) == 4)
        return __uint_as_float(v);
    else
        return __uint_as_float(static_cast<uint32_t>(v) << 16);
}

constexpr int kNT = 128;  // columns n per CTA (4 per lane)
constexpr int kCW = 8;    // output channels per warp
constexpr int kMT = 64;   // output channels per CTA (8 warps)
constexpr int kRC = 32;   // reduction indices per staged chunk (a multiple of G)
constexpr int kXP = kNT + 4;  // padded row of the staged X chunk (16-byte aligned rows)
// shared memory: the X chunk, the chunk's values and rows; reused for the output tile
constexpr int kSmemMain = kRC * kXP * 4 + kMT * kRC * 4 + kMT * kRC;
constexpr int kSmemOut = kNT * (kMT + 1) * 4;
constexpr int kSmem = kSmemMain > kSmemOut ? kSmemMain : kSmemOut;

template <typename TB>
__global__ void __launch_bounds__(256) bbs_gather_kernel(const TB *__restrict__ X, int64_t N, int64_t R,
                                                         const TB *__restrict__ values, const uint8_t *__restrict__ idx,
                                                         int64_t Cout, int G, int K, float *__restrict__ Y,
                                                         uint32_t *status)
{
    __shared__ __align__(16) unsigned char smem[kSmem];
    float(*xs)[kXP] = reinterpret_cast<float(*)[kXP]>(smem);                          // xs[r][n]
    float(*sv)[kRC] = reinterpret_cast<float(*)[kRC]>(smem + kRC * kXP * 4);          // values
    uint8_t(*sr)[kRC] = reinterpret_cast<uint8_t(*)[kRC]>(smem + kRC * kXP * 4 + kMT * kRC * 4);  // rows
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kNT;
    const int64_t co0 = static_cast<int64_t>(blockIdx.y) * kMT;
    const int64_t ng = R / G;
    const int spc = (kRC / G) * K;  // slots per channel in a full chunk
    float acc[kCW][4];
#pragma unroll
    for (int c = 0; c < kCW; ++c)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[c][q] = 0.f;
    bool bad = false;

    for (int64_t r0 = 0; r0 < R; r0 += kRC) {
        const int rc = (R - r0) < kRC ? static_cast<int>(R - r0) : kRC;  // a multiple of G
        __syncthreads();
        for (int e = tid; e < kRC * kNT; e += 256) {
            const int nn = e / kRC, rr = e - nn * kRC;  // consecutive threads: consecutive r
            const int64_t n = n0 + nn;
            xs[rr][nn] = (n < N && rr < rc) ? to_f32(X[n * R + r0 + rr]) : 0.f;
        }
        const int nslots = (rc / G) * K;
        for (int e = tid; e < kMT * spc; e += 256) {
            const int c = e / spc, s = e - c * spc;
            const int64_t co = co0 + c;
            float v = 0.f;
            int row = 0;
            if (co < Cout && s < nslots) {
                const int64_t slot = (co * ng + r0 / G) * K + s;  // group r0/G + s/K, slot s%K
                const int j = idx[slot];
                bad |= j >= G;
                v = to_f32(values[slot]);
                row = (s / K) * G + (j < G ? j : 0);
            }
            sv[c][s] = v;
            sr[c][s] = static_cast<uint8_t>(row);
        }
        __syncthreads();
#pragma unroll
        for (int c = 0; c < kCW; ++c) {
            const int cl = warp * kCW + c;
            for (int s = 0; s < nslots; ++s) {
                const float v = sv[cl][s];
                const float4 x = *reinterpret_cast<const float4 *>(&xs[sr[cl][s]][lane * 4]);
                acc[c][0] = fmaf(v, x.x, acc[c][0]);
                acc[c][1] = fmaf(v, x.y, acc[c][1]);
                acc[c][2] = fmaf(v, x.z, acc[c][2]);
                acc[c][3] = fmaf(v, x.w, acc[c][3]);
            }
        }
    }
    if (bad) report(status, CCI_ERR_INDEX);
    // stage the tile as [n][channel] and write whole rows of channels
    __syncthreads();
    float(*ys)[kMT + 1] = reinterpret_cast<float(*)[kMT + 1]>(smem);
#pragma unroll
    for (int c = 0; c < kCW; ++c)
#pragma unroll
        for (int q = 0; q < 4; ++q) ys[lane * 4 + q][warp * kCW + c] = acc[c][q];
    __syncthreads();
    for (int e = tid; e < kNT * kMT; e += 256) {
        const int nn = e / kMT, c = e - nn * kMT;
        const int64_t n = n0 + nn, co = co0 + c;
        if (n < N && co < Cout) Y[n * Cout + co] = ys[nn][c];
    }
}

}  // namespace bbs

static int grid_of(int64_t total)
{
    const int64_t blocks = (total + 255) / 256;
    return static_cast<int>(blocks < 65536 * 16 ? blocks : 65536 * 16);
}

cudaError_t launch_bbs_pack(const void *W, int dtype, int64_t Cout, int64_t R, int G, int K, void *values,
                            uint8_t *idx, uint32_t *status, cudaStream_t stream)
{
    const int grid = grid_of(Cout * (R / G));
    if (dtype == CCI_F32)
        bbs::bbs_pack_kernel<uint32_t><<<grid, 256, 0, stream>>>(static_cast<const uint32_t *>(W), Cout, R, G, K,
                                                                 static_cast<uint32_t *>(values), idx, status);
    else
        bbs::bbs_pack_kernel<uint16_t><<<grid, 256, 0, stream>>>(static_cast<const uint16_t *>(W), Cout, R, G, K,
                                                                 static_cast<uint16_t *>(values), idx, status);
    return cudaGetLastError();
}

template <typename TB, bool SPLIT, int GC>
static void bbs_decompress_launch(const FwdParams &p, int G, int K, int grid, cudaStream_t stream)
{
    TB *w0 = static_cast<TB *>(const_cast<void *>(p.wdense));
    bbs::bbs_decompress_kernel<TB, SPLIT, GC><<<grid, 256, 0, stream>>>(
        static_cast<const TB *>(p.values), p.idx, p.Cout, p.R, G, K, w0, SPLIT ? w0 + p.Cout * p.R : nullptr,
        p.status);
}

cudaError_t launch_bbs_decompress(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream)
{
    const int grid = grid_of(p.Cout * (p.R / G));
    // the workspace is 16-byte aligned and R is a multiple of G, so every group
    // of G * element size (a multiple of 16) bytes starts 16-byte aligned
    if (dtype == CCI_F32) {
        if (G == 4) bbs_decompress_launch<uint32_t, true, 4>(p, G, K, grid, stream);
        else if (G == 8) bbs_decompress_launch<uint32_t, true, 8>(p, G, K, grid, stream);
        else if (G == 16) bbs_decompress_launch<uint32_t, true, 16>(p, G, K, grid, stream);
        else if (G == 32) bbs_decompress_launch<uint32_t, true, 32>(p, G, K, grid, stream);
        else bbs_decompress_launch<uint32_t, true, 0>(p, G, K, grid, stream);
    } else {
        if (G == 8) bbs_decompress_launch<uint16_t, false, 8>(p, G, K, grid, stream);
        else if (G == 16) bbs_decompress_launch<uint16_t, false, 16>(p, G, K, grid, stream);
        else if (G == 32) bbs_decompress_launch<uint16_t, false, 32>(p, G, K, grid, stream);
        else bbs_decompress_launch<uint16_t, false, 0>(p, G, K, grid, stream);
    }
    return cudaGetLastError();
}

cudaError_t launch_bbs_gather(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream)
{
    const dim3 grid(static_cast<unsigned>((p.N + bbs::kNT - 1) / bbs::kNT),
                    static_cast<unsigned>((p.Cout + bbs::kMT - 1) / bbs::kMT));
    if (dtype == CCI_F32)
        bbs::bbs_gather_kernel<uint32_t><<<grid, 256, 0, stream>>>(static_cast<const uint32_t *>(p.X), p.N, p.R,
                                                                   static_cast<const uint32_t *>(p.values), p.idx,
                                                                   p.Cout, G, K, p.Y, p.status);
    else
        bbs::bbs_gather_kernel<uint16_t><<<grid, 256, 0, stream>>>(static_cast<const uint16_t *>(p.X), p.N, p.R,
                                                                   static_cast<const uint16_t *>(p.values), p.idx,
                                                                   p.Cout, G, K, p.Y, p.status);
    return cudaGetLastError();
}

}  // namespace cci
