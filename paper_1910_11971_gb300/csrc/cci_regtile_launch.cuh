// cci_regtile_launch.cuh -- host launcher of one register-tiled instantiation.
#pragma once

#include "cci_kernels.h"
#include "cci_regtile.cuh"

namespace cci {

inline int device_sm_count()
{
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms > 0 ? sms : 1;
}

template <typename TS, int G, int K, int MG, int T, int D, int WC>
cudaError_t launch_regtile_wc(const FwdParams &p, cudaStream_t stream)
{
    using RT = RegTile<TS, G, K, MG, T, D, WC>;
    static_assert(RT::kTotal <= kMaxSmemPerBlock, "shared-memory layout over the per-block limit");
    auto kern = regtile_kernel<TS, G, K, MG, T, D, WC>;
    static SmemAttrCache attr_cache;
    const cudaError_t attr = smem_attr_once(kern, static_cast<int>(RT::kTotal), attr_cache);
    if (attr != cudaSuccess) return attr;
    const int64_t groups = p.Cout / G;
    const int64_t n_ct = (groups + RT::kNGR - 1) / RT::kNGR;
    const int64_t n_nt = (p.N + RT::kNTC - 1) / RT::kNTC;
    const int64_t n_tiles = n_ct * n_nt;
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, RT::kThreads, RT::kTotal);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t resident = static_cast<int64_t>(device_sm_count()) * per_sm;
    const unsigned grid = static_cast<unsigned>(n_tiles < resident ? n_tiles : resident);
    kern<<<grid, RT::kThreads, RT::kTotal, stream>>>(p, n_ct, n_tiles);
    return cudaGetLastError();
}

template <typename TS, int G, int K, int MG, int T, int D>
cudaError_t launch_regtile(const FwdParams &p, cudaStream_t stream)
{
    if (regtile_wc(p.Cout / G, MG) == 8) return launch_regtile_wc<TS, G, K, MG, T, D, 8>(p, stream);
    return launch_regtile_wc<TS, G, K, MG, T, D, 4>(p, stream);
}

}  // namespace cci

// table row for one instantiation (dtype tag, storage type, G, K, MG, T, D)
#define CCI_REGTILE_ROW(DT, TS, G, K, MG, T, D)                                                    \
    {DT, G, K, MG, T, D, (D == 0 ? "expand_" #TS "_G" #G "_K" #K "_MG" #MG "_T" #T                  \
                                 : "regtile_" #TS "_G" #G "_K" #K "_MG" #MG "_T" #T "_D" #D),       \
     &cci::launch_regtile<TS, G, K, MG, T, D>},
