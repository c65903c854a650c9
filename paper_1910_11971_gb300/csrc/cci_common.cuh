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
