// cci_common.cuh -- device helpers shared by the libcci kernels (sm_103a).
#pragma once

#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "cci.h"

namespace cci {

// Argument block of the forward products.  A product is the convolution with
// H = W = KH = KW = 1, so both entry points share one parameter set:
//   column n = (b, p, q), reduction index r = (kh*KW + kw)*Cin + ci.
struct FwdParams {
    const void *X;
    const void *values;
    const uint8_t *idx;
    float *Y;            // fp32 output, or bf16 when out_bf16
    uint32_t *status;
    int64_t N;      // columns = B*P*Q
    int64_t Cout;
    int64_t R;      // Cin*KH*KW
    int64_t Cin;
    int64_t H, W;   // input image (1 x 1 for a product)
    int64_t P, Q;   // output image (1 x 1 for a product)
    int KH, KW, sh, sw, ph, pw;
    int is_conv;
    const void *wdense;  // dense decompressed weights [Cout][R] (workspace kernels only)
    int G, K;            // group size and kept weights per group (fused tensor-core kernel)
    // output epilogue (workspace kernels only): y + bias[co], ReLU, bf16 output
    const float *bias;   // nullptr: none
    int relu;
    int out_bf16;        // Y holds bf16 (round to nearest even) instead of fp32
    int kin;             // workspace kernels: reduction indices copied per stage (bf16
                         // products with R < 64: R rounded up to 16; else the whole stage)
};

__device__ __forceinline__ void report(uint32_t *status, cci_status code)
{
    if (status) atomicOr(status, 1u << static_cast<unsigned>(code));
}

// bf16 bits -> fp32 value (exact: bf16 is the upper half of a binary32)
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t b16)
{
    return __uint_as_float(b16 << 16);
}

// ---- fp32 operands of the tensor-core product ----
// An fp32 value v is split as v = hi + lo: hi is a tf32 value (fp32 bits whose
// low 13 mantissa bits are zero), lo = v - hi exactly.  Per 32 reduction indices
// the product takes three terms, 8 MMAs in all (x: activation, w: weight):
//   hi(x) * hi(w)                 tf32, 4 MMAs of 8 indices (exact products)
//   bf16(x) * bf16(lo(w))         bf16, 2 MMAs of 16 indices
//   bf16(lo(x)) * bf16(hi(w))     bf16, 2 MMAs of 16 indices
// The first cross term takes the whole x, so lo(x) * lo(w) is included.  Weight
// hi is the nearest tf32 (|lo| <= 2^-11 |w|); activation hi is truncated (|lo| <
// 2^-10 |x|, one logic op in the producers); bf16 conversions round to nearest
// and saturate to the largest finite bf16.  Per term of the reduction the error
// is at most |x||w| (2^-8 * 2^-11 + 2^-8 * 2^-10 (1 + 2^-11)), about
// 5.7e-6 |x||w|, under the 1e-5 sum |x||w| tolerance before the fp32 accumulation.
// Operand planes (weights in the workspace; activations in shared or tensor
// memory): plane 0 holds hi as fp32 bits, [rows][R]; plane 1 holds bf16 pairs
// [rows][ceil(R / 32) * 64]: for chunk c of 32 indices, element c * 64 + t is the
// first bf16 operand of index c * 32 + t (t < 32) and element c * 64 + 32 + t
// the second (bf16(hi(w)) and bf16(lo(w)) for weights, bf16(x) and bf16(lo(x))
// for activations); indices past R hold zeros.
__device__ __forceinline__ uint32_t tf32_trunc(uint32_t v) { return v & 0xffffe000u; }

// nearest tf32 (ties to even); a finite value that would round up into the
// exponent of inf keeps its truncation, inf and NaN are truncated
__device__ __forceinline__ uint32_t tf32_rn(uint32_t v)
{
    const uint32_t r = (v + 0x0fffu + ((v >> 13) & 1u)) & 0xffffe000u;
    return (r & 0x7f800000u) == 0x7f800000u ? (v & 0xffffe000u) : r;
}

// bf16 pair (e0 in the low half), round to nearest, saturating at the largest
// finite bf16
__device__ __forceinline__ uint32_t bf16x2_rn_sat(float e0, float e1)
{
    uint32_t r;
    asm("cvt.rn.satfinite.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(e1), "f"(e0));
    return r;
}

// 16-bit elements of plane 1 per row for R reduction indices
__device__ __forceinline__ int64_t split_plane1_row(int64_t R) { return (R + 31) / 32 * 64; }

// writes weights w[0..3] of row `row` at indices r0 .. r0 + 3 (r0 % 4 == 0) into
// the two weight planes; the writer of the last indices (r0 + 4 == R) also
// zeroes the rest of plane 1's last chunk
__device__ __forceinline__ void store_w_split4(uint32_t *plane0, uint16_t *plane1, int64_t R, int64_t row,
                                               int64_t r0, const uint32_t (&w)[4])
{
    uint32_t h[4];
    float l[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        h[e] = tf32_rn(w[e]);
        l[e] = __uint_as_float(w[e]) - __uint_as_float(h[e]);
    }
    __stcg(reinterpret_cast<uint4 *>(plane0 + row * R + r0), make_uint4(h[0], h[1], h[2], h[3]));
    uint16_t *q = plane1 + row * split_plane1_row(R) + (r0 >> 5) * 64 + (r0 & 31);
    __stcg(reinterpret_cast<uint2 *>(q), make_uint2(bf16x2_rn_sat(__uint_as_float(h[0]), __uint_as_float(h[1])),
                                                    bf16x2_rn_sat(__uint_as_float(h[2]), __uint_as_float(h[3]))));
    __stcg(reinterpret_cast<uint2 *>(q + 32), make_uint2(bf16x2_rn_sat(l[0], l[1]), bf16x2_rn_sat(l[2], l[3])));
    if (r0 + 4 == R && (R & 31) != 0) {
        for (int t = static_cast<int>(R & 31); t < 32; t += 4) {
            uint16_t *z = plane1 + row * split_plane1_row(R) + (r0 >> 5) * 64 + t;
            __stcg(reinterpret_cast<uint2 *>(z), make_uint2(0u, 0u));
            __stcg(reinterpret_cast<uint2 *>(z + 32), make_uint2(0u, 0u));
        }
    }
}

// the same for one weight at any index r (2-byte plane-1 stores); the writer of
// index R - 1 zeroes the rest of the last chunk
__device__ __forceinline__ void store_w_split1(uint32_t *plane0, uint16_t *plane1, int64_t R, int64_t row,
                                               int64_t r, uint32_t w)
{
    const uint32_t h = tf32_rn(w);
    const float l = __uint_as_float(w) - __uint_as_float(h);
    plane0[row * R + r] = h;
    uint16_t *q = plane1 + row * split_plane1_row(R) + (r >> 5) * 64;
    q[r & 31] = static_cast<uint16_t>(bf16x2_rn_sat(__uint_as_float(h), 0.0f));
    q[32 + (r & 31)] = static_cast<uint16_t>(bf16x2_rn_sat(l, 0.0f));
    if (r == R - 1)
        for (int t = static_cast<int>((r & 31) + 1); t < 32; ++t) q[t] = q[32 + t] = 0;
}

// Packed fp32 FMA on two lanes: d = a * b + d, element-wise on (lo, hi) pairs,
// each element an IEEE binary32 fused multiply-add with one rounding.
__device__ __forceinline__ void ffma2(unsigned long long &d, unsigned long long a,
                                      unsigned long long b)
{
    asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(d) : "l"(a), "l"(b));
}

__device__ __forceinline__ unsigned long long pack2(float lo, float hi)
{
    return (static_cast<unsigned long long>(__float_as_uint(hi)) << 32) |
           static_cast<unsigned long long>(__float_as_uint(lo));
}

__device__ __forceinline__ float lo_of(unsigned long long v)
{
    return __uint_as_float(static_cast<uint32_t>(v));
}

__device__ __forceinline__ float hi_of(unsigned long long v)
{
    return __uint_as_float(static_cast<uint32_t>(v >> 32));
}

// Output pixel of column n and the first input pixel of its receptive field.
struct ColumnSite {
    int64_t img;   // offset of image b in X (elements): b*H*W*Cin
    int hb, wb;    // p*sh - ph, q*sw - pw
};

__device__ __forceinline__ ColumnSite column_site(const FwdParams &p, int64_t n)
{
    ColumnSite s;
    if (!p.is_conv) {  // a product: column n is row n of X, no receptive field
        s.img = n * p.Cin;
        s.hb = 0;
        s.wb = 0;
        return s;
    }
    const int64_t pq = p.P * p.Q;
    const int64_t b = n / pq;
    const int64_t rem = n - b * pq;
    const int64_t op = rem / p.Q;
    const int64_t oq = rem - op * p.Q;
    s.img = b * p.H * p.W * p.Cin;
    s.hb = static_cast<int>(op * p.sh - p.ph);
    s.wb = static_cast<int>(oq * p.sw - p.pw);
    return s;
}

// Element offset in X of x[n][r] for column site s, or -1 outside the image.
// r must be < R.
__device__ __forceinline__ int64_t x_offset(const FwdParams &p, const ColumnSite &s, int64_t r)
{
    const int64_t tap = r / p.Cin;
    const int64_t ci = r - tap * p.Cin;
    const int kh = static_cast<int>(tap / p.KW);
    const int kw = static_cast<int>(tap - static_cast<int64_t>(kh) * p.KW);
    const int h = s.hb + kh;
    const int w = s.wb + kw;
    if (h < 0 || h >= p.H || w < 0 || w >= p.W) return -1;
    return s.img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
}

// Per-device record of a kernel's dynamic shared-memory limit: the CUDA runtime
// keeps cudaFuncAttributeMaxDynamicSharedMemorySize per device context, so it is
// set once on every device the kernel is launched on (the first launch there).
struct SmemAttrCache {
    static constexpr int kDevices = 64;
    std::mutex m;
    bool set[kDevices] = {};
    cudaError_t err[kDevices] = {};
};

// cudaFuncSetAttribute(kern, MaxDynamicSharedMemorySize, bytes) on the current
// device, once per device; later calls return the first call's result
template <typename Kern>
cudaError_t smem_attr_once(Kern kern, int bytes, SmemAttrCache &c)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= SmemAttrCache::kDevices)
        return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(c.m);
    if (!c.set[dev]) {
        c.err[dev] = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        c.set[dev] = true;
    }
    return c.err[dev];
}

}  // namespace cci
