// Internal interface between the host core (cm_host.cpp) and the byte-comparison
// kernels of the optional re-delivery fast path (dedup.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace cm {

constexpr int kMaxComparePairs = 128;         // pairs per launch
constexpr uint64_t kCompareChunkVecs = 2048;   // 16-byte vectors of each array per chunk

// Two fragments of one shape: the K and V arrays of a delivery (a) and of a candidate (b),
// each `vecs` 16-byte vectors long. All four pointers are 16-byte aligned.
struct ComparePair {
    const uint4 *a_k, *a_v, *b_k, *b_v;
    uint64_t vecs;
};

struct CompareLaunch {
    uint32_t count;                               // pairs, <= kMaxComparePairs
    uint32_t pad_;
    // prefix sums of the pairs' chunk counts: 2 ceil(vecs / kCompareChunkVecs) per pair
    uint64_t chunk_begin[kMaxComparePairs + 1];
    ComparePair pair[kMaxComparePairs];
    uint32_t *differ;                             // device, one word per pair, zeroed before
};

// differ[p] |= 1 if the first 4 KiB of the pair's K arrays differ (one block per pair).
cudaError_t launch_compare_prefix(const CompareLaunch &c, cudaStream_t stream);

// differ[p] |= 1 if the pair's K or V arrays differ anywhere (a persistent grid over all
// chunks of all pairs; the chunks of a pair already found to differ are skipped).
cudaError_t launch_compare_full(const CompareLaunch &c, int num_sms, cudaStream_t stream);

}  // namespace cm
