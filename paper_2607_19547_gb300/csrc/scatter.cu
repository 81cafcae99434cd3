// Scatter-back of repaired rows (ChronoStitch Sec. 2): the fresh keys and
// values of the recomputed tokens replace their stored rows in the composed
// cache before each layer's attention.  An indexed copy, HBM-bound: one row
// read and one row written per (layer, repaired token).
//
// One warp per (layer, row), 16-byte accesses, lanes striding over the row; a
// grid-stride loop covers every (layer, row).  The destination token comes from
// idx; an index outside [0, T) skips the row and records CS_ERR_DEVICE_ARG.
#include "cs_device.cuh"
#include "cs_internal.h"

#include <algorithm>

namespace cs {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

__global__ void __launch_bounds__(kThreads)
scatter_kernel(uint4 *__restrict__ cache, const uint4 *__restrict__ rows, int n_layers, int T,
               long long cache_stride16, int n_rows, long long rows_stride16, int row16,
               const int *__restrict__ idx, unsigned int *status) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const long long total = static_cast<long long>(n_layers) * n_rows;
    for (long long w = static_cast<long long>(blockIdx.x) * kWarps + (threadIdx.x >> 5); w < total;
         w += static_cast<long long>(gridDim.x) * kWarps) {
        const int l = static_cast<int>(w / n_rows), r = static_cast<int>(w - static_cast<long long>(l) * n_rows);
        const int d = __ldg(idx + r);
        if (d < 0 || d >= T) {
            if (lane == 0 && l == 0) report_error(status, 5u, kSiteScatter, static_cast<unsigned>(r));
            continue;
        }
        const uint4 *src = rows + l * rows_stride16 + static_cast<long long>(r) * row16;
        uint4 *dst = cache + l * cache_stride16 + static_cast<long long>(d) * row16;
        for (int i = lane; i < row16; i += 32) dst[i] = __ldcs(src + i);
    }
}

}  // namespace

cudaError_t launch_scatter(void *cache, const void *rows, int n_layers, int T, long long cache_stride16,
                           int n_rows, long long rows_stride16, int row16, const int *idx,
                           unsigned int *status, cudaStream_t s) {
    const long long warps = static_cast<long long>(n_layers) * n_rows;
    if (warps == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const long long want = (warps + kWarps - 1) / kWarps;
    const int grid = static_cast<int>(std::min<long long>(want, static_cast<long long>(sms) * 16));
    return launch_pdl(scatter_kernel, dim3(grid), dim3(kThreads), 0, s, static_cast<uint4 *>(cache),
                      static_cast<const uint4 *>(rows), n_layers, T, cache_stride16, n_rows,
                      rows_stride16, row16, idx, status);
}

}  // namespace cs
