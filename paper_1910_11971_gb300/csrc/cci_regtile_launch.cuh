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

template <typename TS, int G, int K, int MG, int T>
cudaError_t launch_regtile(const FwdParams &p, cudaStream_t stream)
{
    using RT = RegTile<TS, G, K, MG, T>;
    auto kern = regtile_kernel<TS, G, K, MG, T>;
    // opt in to the largest layout any channel split uses, once per process
    static const cudaError_t attr = [kern] {
        const size_t most = RT::layout(4).total > RT::layout(8).total ? RT::layout(4).total : RT::layout(8).total;
        if (most > kMaxSmemPerBlock) return cudaErrorInvalidConfiguration;
        return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(most));
    }();
    if (attr != cudaSuccess) return attr;
    const int64_t groups = p.Cout / G;
    const int wc = regtile_wc(groups, MG);
    const auto L = RT::layout(wc);
    if (L.total > kMaxSmemPerBlock) return cudaErrorInvalidConfiguration;
    const int64_t n_ct = (groups + L.ngroups - 1) / L.ngroups;
    const int64_t n_nt = (p.N + L.ntc - 1) / L.ntc;
    const int64_t n_tiles = n_ct * n_nt;
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, RT::kThreads, L.total);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int64_t resident = static_cast<int64_t>(device_sm_count()) * per_sm;
    const unsigned grid = static_cast<unsigned>(n_tiles < resident ? n_tiles : resident);
    kern<<<grid, RT::kThreads, L.total, stream>>>(p, wc, n_ct, n_tiles);
    return cudaGetLastError();
}

}  // namespace cci

// table row for one instantiation (dtype tag, storage type, G, K, MG, T)
#define CCI_REGTILE_ROW(DT, TS, G, K, MG, T)                                                       \
    {DT, G, K, MG, T, "regtile_" #TS "_G" #G "_K" #K "_MG" #MG "_T" #T,                             \
     &cci::launch_regtile<TS, G, K, MG, T>},
