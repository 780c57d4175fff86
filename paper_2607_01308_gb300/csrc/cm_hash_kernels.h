// Internal interface between the host core (cm_host.cpp) and the content-address
// kernels (blake2s_tree.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "cm.h"

namespace cm {

// ---------------------------------------------------------------- content address
// BLAKE2s tree mode (RFC 7693 compression; tree parameters of the BLAKE2 paper):
// 1024-byte leaves, fanout 16, 16-byte node digests.
constexpr int kDigestBytes = 16;
constexpr int kLeafBytes = 1024;
constexpr int kFanout = 16;

// Chaining value a node starts from: IV xor the 32-byte parameter block with the
// node offset and node depth fields zero. Kernels xor in offset and depth.
struct TreeParams {
    uint32_t h_base[8];
};

struct LeafLaunch {
    const uint8_t *k;              // fragment K, device
    const uint8_t *v;              // fragment V, device
    uint64_t plane_bytes;          // bytes of one layer of K (= of V): H*T*d*2
    uint64_t stream_bytes;         // 2 * L * plane_bytes
    uint64_t num_leaves;           // ceil(stream_bytes / 1024)
    uint64_t norm_begin;           // stream offset of K[l*]; its length is plane_bytes
    uint32_t row_bytes;            // d*2; a power of two in [32, 1024]
    uint32_t seq_len;              // T
    unsigned long long *norm_key;  // Q[T] accumulators, zeroed before the launch
    uint8_t *digests;              // num_leaves * 16 bytes out
    TreeParams tree;
};

// Level 0 of up to kMaxLeafGroup fragments in one launch: one thread per leaf, the
// leaf blocks of fragment i being [block_begin[i], block_begin[i + 1]) (set by the
// caller); after the last leaf block, one thread per row of K[l*] for the routing-layer
// norm key, the norm blocks of fragment i being block_begin[count] +
// [norm_block_begin[i], norm_block_begin[i + 1]) (set by the launcher).
constexpr int kMaxLeafGroup = 32;
constexpr int kLeafBlockThreads = 128;   // threads (= leaves or rows) per block of the leaf launch
struct LeafGroup {
    uint32_t count;
    uint32_t pad_;
    uint64_t block_begin[kMaxLeafGroup + 1];
    uint64_t norm_block_begin[kMaxLeafGroup + 1];
    LeafLaunch frag[kMaxLeafGroup];
};
// kBoth: leaves and norm keys in one launch; kLeaves / kNormKeys: one of the two (the
// norm keys alone read only K[l*], 1/(2L) of the bytes).
enum class LeafPhases { kBoth, kLeaves, kNormKeys };
cudaError_t launch_leaf_hash_group(const LeafGroup &g, cudaStream_t stream, LeafPhases phases);
// Leaf-hash blocks that fit on one SM at once (occupancy of leaf_hash_kernel), or 0 on error.
int leaf_hash_blocks_per_sm();

// Level 0 of one fragment (a group of one).
cudaError_t launch_leaf_hash(const LeafLaunch &a, cudaStream_t stream);

// Level `depth` >= 1: node j hashes the digests of children [16 j, 16 j + 16).
cudaError_t launch_inner_hash(const uint8_t *children, uint64_t num_children, uint8_t *out,
                              uint64_t num_nodes, uint32_t depth, const TreeParams &tree,
                              cudaStream_t stream);

constexpr int kMaxGroup = 32;

// Every tree level above the leaves, for up to kMaxGroup fragments. One thread per
// level-s node hashes it; then, level by level, the thread that completes a parent's
// last child (a per-node arrival counter, zeroed before the launch) hashes that parent,
// up to the root. No thread ever waits for another. With fewer than kSplitLevel1Nodes
// level-1 nodes in all, one launch with s = 1. With more, a first launch hashes level 1
// with every lane of a warp busy and many warps per SM, and a second runs the scheme
// above with s = 2 (in one launch, each warp would hash 32 level-1 nodes and then two
// level-2 parents with two of its lanes). The caller sets node_begin from the level-1
// sizes.
constexpr int kMaxLevels = 12;
struct TreeTopFragment {
    uint8_t *level[kMaxLevels];       // digests of level k; level[levels - 1] is the root
    uint64_t size[kMaxLevels];        // nodes of level k
    uint32_t *arrivals[kMaxLevels];   // per node of level k >= 2: children finished so far
    uint32_t levels;                  // >= 2
    TreeParams tree;
};
struct TreeTop {
    uint32_t count;
    uint64_t node_begin[kMaxGroup + 1];   // prefix sum of the fragments' level-1 sizes (level 2 in the second launch)
    TreeTopFragment frag[kMaxGroup];
};
constexpr uint64_t kSplitLevel1Nodes = 32768;
cudaError_t launch_tree_top(const TreeTop &t, cudaStream_t stream);
int tree_top_kernels(const TreeTop &t);   // kernels launch_tree_top launches for t

// *flag |= 1 if the `bytes` bytes at a and b differ (16-byte aligned, bytes % 16 == 0).
cudaError_t launch_compare(const void *a, const void *b, uint64_t bytes, unsigned int *flag,
                           cudaStream_t stream);

// Bounds-checked builds: reads and zeroes the content-address kernels' violation count on
// the current device (0 in other builds).
cudaError_t take_hash_bounds_violations(unsigned int *out);

// Host-core helpers used by the allocation-free entry point in blake2s_tree.cu.
TreeParams make_tree_params(int32_t L, int32_t H, int32_t d, int32_t T);
cm_status check_fragment(const cm_fragment *f);
cm_status report_error(cm_status st, const char *msg);

}  // namespace cm
