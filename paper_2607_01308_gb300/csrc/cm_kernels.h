// Internal interface between the host core (cm_host.cpp) and the CUDA kernels
// (blake2s_tree.cu, render.cu). Not part of the public ABI.
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
    uint32_t row_bytes;            // d*2; a power of two <= 1024, so rows never straddle leaves
    uint32_t seq_len;              // T
    unsigned long long *norm_key;  // Q[T] accumulators, zeroed before the launch
    uint8_t *digests;              // num_leaves * 16 bytes out
    TreeParams tree;
};

// Level 0: one thread per leaf; also accumulates the routing-layer norm key.
cudaError_t launch_leaf_hash(const LeafLaunch &a, cudaStream_t stream);

// Level `depth` >= 1: node j hashes the digests of children [16 j, 16 j + 16).
cudaError_t launch_inner_hash(const uint8_t *children, uint64_t num_children, uint8_t *out,
                              uint64_t num_nodes, uint32_t depth, const TreeParams &tree,
                              cudaStream_t stream);

constexpr int kMaxGroup = 32;

// Every tree level above the leaves, for up to kMaxGroup fragments, in one launch.
// One thread per level-1 node hashes it; then, level by level, the thread that
// completes a parent's last child (a per-node arrival counter, zeroed before the
// launch) hashes that parent, up to the root. No thread ever waits for another.
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
    uint64_t node_begin[kMaxGroup + 1];   // prefix sum of the fragments' level-1 sizes
    TreeTopFragment frag[kMaxGroup];
};
cudaError_t launch_tree_top(const TreeTop &t, cudaStream_t stream);

// *flag |= 1 if the `bytes` bytes at a and b differ (16-byte aligned, bytes % 16 == 0).
cudaError_t launch_compare(const void *a, const void *b, uint64_t bytes, unsigned int *flag,
                           cudaStream_t stream);

// Host-core helpers used by the allocation-free entry point in blake2s_tree.cu.
TreeParams make_tree_params(int32_t L, int32_t H, int32_t d, int32_t T);
cm_status check_fragment(const cm_fragment *f);
cm_status report_error(cm_status st, const char *msg);

// ---------------------------------------------------------------- render
constexpr int kMaxSlots = 32;          // fragments per render launch
constexpr int kMaxTablePairs = 1792;   // sum over slots of head_dim / 2
constexpr int kChunkBytes = 4096;      // bytes of one source plane handled per work item

struct RenderSlot {
    const void *k;              // source K [L][H][T][d], device
    const void *v;              // source V
    void *k_out;                // contiguous output of the slot's set, [L][H][capacity][d]
    void *v_out;                // (unused for paged outputs)
    int64_t capacity;           // token rows per (layer, head) plane of k_out / v_out
    int64_t seq_len;            // T
    int64_t offset;             // s: first output position of this slot
    uint32_t chunk_begin;       // first global work item of this slot
    uint32_t chunks_per_plane;  // ceil(T / rows_per_chunk)
    int32_t rotate;             // 0: K is copied as bytes (offset 0)
    int32_t table_base;         // index of (cos, sin)[j = 0] of this slot in cs[]
};

// Passed by value (kernel parameter space, < 32 KiB), so a launch owns its table.
struct RenderParams {
    void *k_pool;               // paged outputs only: the block pools (see below)
    void *v_pool;
    int32_t num_layers;
    int32_t num_heads;
    int32_t head_dim;
    int32_t num_slots;
    int32_t rows_per_chunk;     // kChunkBytes / (2 d)
    int32_t log2_pairs_per_row; // log2(d / 16)
    uint32_t total_chunks;
    uint32_t pad_;
    unsigned int *error;        // device word: bit 0 set when a bounded wait timed out
    uint32_t withhold_warp;     // failure-injection hook: global warp index + 1 whose first
                                // TMA load is never issued (its wait runs out); 0 = none
    int32_t paged;              // 1: outputs are block pools addressed through block_table
    // paged output: token pos of (layer l, head h) lives at pool + block_table[pos / block_size]
    // * stride_block + l * stride_layer + h * stride_head + (pos % block_size) * stride_token
    // (element strides, head_dim contiguous)
    const int32_t *block_table; // device
    int64_t block_size;
    int32_t log2_block_size;    // >= 0 when block_size is a power of two, else -1
    int32_t pad3_;
    int64_t stride_block, stride_layer, stride_head, stride_token;
    RenderSlot slot[kMaxSlots];
    double cs[2 * kMaxTablePairs];   // (cos a, sin a) of a = s * theta^(-2j/d), interleaved
};

// One CTA of `warps` warps (16, or 8 to leave half of each SM's registers to kernels of
// other streams) per SM; render_prepare() once per device before the first launch.
cudaError_t launch_render(const RenderParams &p, int grid, int warps, cudaStream_t stream);
cudaError_t render_prepare();

}  // namespace cm
