// cci_dense_tc.cu -- the one-pass decompression of the packed weights into the
// workspace of CCI_ALGO_DENSE_TC_WS (namespace dc), which precedes the
// workspace GEMM, and the diagnostic of the kernels' bounded waits.
#include "cci_gemm_ws.cuh"

namespace cci {
namespace tc {

// Diagnostic of the bounded waits of the tensor-core kernels: one thread initialises an mbarrier that
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
// layers its two operand planes (store_w_split4: hi as a tf32 value, then the
// bf16 pairs of hi and lo per 32-wide chunk) for the product
// hi(x) hi(w) + bf16(x) bf16(lo(w)) + bf16(lo(x)) bf16(hi(w)).
// One block per (group gi, slab of kSlab columns r): each thread scatters the K
// kept weights of one column into a zeroed [G][kSlab] tile in shared memory,
// then the block writes the G rows of the slab with 16-byte stores.  Index sets
// must be strictly increasing (as cci_pack writes them); anything else is
// reported as CCI_ERR_INDEX.
// ===========================================================================
namespace dc {

// a launch as a programmatic dependent of the previous kernel on the stream: it
// may be scheduled while that kernel finishes (the kernel itself waits for it
// with griddepcontrol.wait before touching memory)
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute la[1];
    la[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    la[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = la;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

constexpr int kSlab = 256;  // columns r per block (= threads per block)

// T = uint16_t (bf16 bits) or uint32_t (fp32 bits); SPLIT: write the two operand
// planes (fp32 only: plane 0 at w0, plane 1 at w1), else the weights to w0.  R
// must be a multiple of the elements per 16 bytes.
template <typename T, int G, int K, bool SPLIT>
__global__ void __launch_bounds__(kSlab) decompress_kernel(const T *__restrict__ values,
                                                           const uint8_t *__restrict__ idx, int64_t R,
                                                           int64_t slabs, T *__restrict__ w0, T *__restrict__ w1,
                                                           uint32_t *status)
{
    constexpr int V = 16 / static_cast<int>(sizeof(T));  // elements per 16-byte store
    __shared__ __align__(16) T tile[G][kSlab];
    // launched as a programmatic dependent of the kernel before it (the pack):
    // nothing is read or written before that grid has completed
    asm volatile("griddepcontrol.wait;" ::: "memory");
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
            const uint32_t w[4] = {x.x, x.y, x.z, x.w};
            store_w_split4(reinterpret_cast<uint32_t *>(w0), reinterpret_cast<uint16_t *>(w1), R, gi * G + j, rr, w);
        } else {
            __stcg(reinterpret_cast<uint4 *>(w0 + off), x);
        }
    }
}

// bf16 form without shared memory: each thread expands an item of 8 output
// channels x 8 reduction indices from its group's packed runs in registers (the
// expansion of the fused GEMM's producers) and writes the 8 rows with 16-byte
// stores; blocks run along r (coalesced rows), the block's y index is the row
// block, so no thread divides.  Index sets are checked everywhere.  Needs
// G in {4, 8, 16, 32}, K in {1, 2, 4, 8}, K <= G / 2, R % 8 == 0, 16-byte
// aligned packed arrays and workspace, Cout / 8 <= 65535.
template <int K>
__global__ void __launch_bounds__(128) decompress_rows_kernel(FwdParams p, uint16_t *__restrict__ w0)
{
    asm volatile("griddepcontrol.wait;" ::: "memory");  // as decompress_kernel
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) * 8;
    if (r >= p.R) return;
    const int64_t co = static_cast<int64_t>(blockIdx.y) * 8;
    const int lg = 31 - __clz(p.G);
    const int64_t groups = p.Cout / p.G;
    const int64_t g = co >> lg;
    const int j0 = static_cast<int>(co & (p.G - 1));
    ws::pk::Runs<K> run;
    ws::pk::load_item<K>(run, p, g, r, groups);
    uint32_t out[8][4];
    bool bad = false;
    ws::pk::expand_item<K>(out, run, p.G, g, j0, groups, 8, true, bad);
    if (bad) report(p.status, CCI_ERR_INDEX);
#pragma unroll
    for (int jj = 0; jj < 8; ++jj)
        if (co + jj < p.Cout)
            __stcg(reinterpret_cast<uint4 *>(w0 + (co + jj) * p.R + r),
                   make_uint4(out[jj][0], out[jj][1], out[jj][2], out[jj][3]));
}

bool rows_ok(const FwdParams &p, int G, int K)
{
    return (G == 4 || G == 8 || G == 16 || G == 32) && (K == 1 || K == 2 || K == 4 || K == 8) && 2 * K <= G &&
           p.R % 8 == 0 && (p.Cout + 7) / 8 <= 65535 && (p.R / 8 + 127) / 128 <= 0x7fffffff &&
           reinterpret_cast<uintptr_t>(p.values) % 16 == 0 && reinterpret_cast<uintptr_t>(p.idx) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(p.wdense) % 16 == 0;
}

template <typename T, int G, int K, bool SPLIT>
cudaError_t launch(const FwdParams &p, cudaStream_t stream)
{
    if constexpr (!SPLIT) {
        if (rows_ok(p, G, K) && K <= 8) {
            FwdParams q = p;
            q.G = G;
            q.K = K;
            const dim3 grid(static_cast<unsigned>((p.R / 8 + 127) / 128), static_cast<unsigned>((p.Cout + 7) / 8));
            return launch_pdl(decompress_rows_kernel<(K <= 8 ? K : 8)>, grid, dim3(128), stream, q,
                              static_cast<uint16_t *>(const_cast<void *>(p.wdense)));
        }
    }
    const int64_t slabs = (p.R + kSlab - 1) / kSlab;
    const int64_t blocks = (p.Cout / G) * slabs;
    if (blocks > 0x7fffffff) return cudaErrorInvalidValue;
    T *w0 = static_cast<T *>(const_cast<void *>(p.wdense));
    T *w1 = SPLIT ? w0 + p.Cout * p.R : nullptr;
    return launch_pdl(decompress_kernel<T, G, K, SPLIT>, dim3(static_cast<unsigned>(blocks)), dim3(kSlab), stream,
                      static_cast<const T *>(p.values), p.idx, p.R, slabs, w0, w1, p.status);
}

}  // namespace dc

// (G, K) pairs of the workspace family: decompression into p.wdense, then the GEMM
cudaError_t launch_dense_tc_ws(const FwdParams &p, int dtype, int G, int K, cudaStream_t stream)
{
#define CCI_TC_CASE(g, k)                                                                   \
    if (G == g && K == k) {                                                                 \
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

namespace dc {

// one thread per 4 consecutive r of one row: the dense weights into the planes
__global__ void __launch_bounds__(256) dense_split_kernel(const uint32_t *__restrict__ W, int64_t Cout, int64_t R,
                                                          uint32_t *plane0, uint16_t *plane1)
{
    const int64_t q = R / 4;
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < Cout * q;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t row = t / q, r0 = (t - row * q) * 4;
        const uint4 x = __ldg(reinterpret_cast<const uint4 *>(W + row * R + r0));
        const uint32_t w[4] = {x.x, x.y, x.z, x.w};
        store_w_split4(plane0, plane1, R, row, r0, w);
    }
}

}  // namespace dc

cudaError_t launch_dense_split(const uint32_t *W, int64_t Cout, int64_t R, void *planes, cudaStream_t stream)
{
    uint32_t *p0 = static_cast<uint32_t *>(planes);
    uint16_t *p1 = reinterpret_cast<uint16_t *>(p0 + Cout * R);
    const int64_t work = Cout * (R / 4);
    const int64_t blocks = (work + 255) / 256;
    dc::dense_split_kernel<<<static_cast<unsigned>(blocks < 65536 ? blocks : 65536), 256, 0, stream>>>(W, Cout, R, p0,
                                                                                                      p1);
    return cudaGetLastError();
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
