// Small device-to-host results (content addresses and norm keys, comparison flags, the
// error word) written by the SMs straight into pinned host memory through its
// device-mapped address. A copy engine serves its copies in order, so a few hundred
// bytes queued behind a multi-gigabyte device-to-host copy of another stream (the
// previous merge's cache going out) would wait for that copy to finish; stores from a
// kernel travel the host link without waiting for it.
#include "cm_readback_kernels.h"

namespace cm {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
readback_kernel(uint32_t *__restrict__ dst, const uint32_t *__restrict__ src, uint64_t words) {
    for (uint64_t i = (uint64_t)blockIdx.x * kThreads + threadIdx.x; i < words;
         i += (uint64_t)gridDim.x * kThreads)
        dst[i] = __ldcg(src + i);
}

}  // namespace

cudaError_t launch_readback(void *host_mapped_dst, const void *src, size_t bytes,
                            cudaStream_t stream) {
    const uint64_t words = bytes / 4;
    if (words == 0) return cudaSuccess;
    uint64_t blocks = (words + kThreads - 1) / kThreads;
    if (blocks > 256) blocks = 256;
    readback_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(
        static_cast<uint32_t *>(host_mapped_dst), static_cast<const uint32_t *>(src), words);
    return cudaGetLastError();
}

}  // namespace cm
