// Internal interface between the host core (cm_host.cpp) and the render kernel
// (render.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "cm.h"

namespace cm {

// ---------------------------------------------------------------- render
constexpr int kMaxSlots = 32;          // fragments per render launch
constexpr int kMaxTablePairs = 1792;   // sum over slots of head_dim / 2

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
    int32_t rows_per_chunk;     // render_item_bytes(width) / (2 d)
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
    int64_t table_entries;      // entries of block_table (bounds-checked builds check reads)
    int64_t stride_block, stride_layer, stride_head, stride_token;
    RenderSlot slot[kMaxSlots];
    double cs[2 * kMaxTablePairs];   // (cos a, sin a) of a = s * theta^(-2j/d), interleaved
};

// How much of each SM a render takes:
//   kFull         the register kernel, 3 CTAs of 8 warps per SM (cm_context_set_render_warps(16),
//                 the default): the fastest render alone
//   kHalf         the TMA kernel, one CTA of 8 warps (3 stages each) per SM
//                 (cm_context_set_render_warps(8)): half of each SM's registers stay free for
//                 kernels of other streams
//   kBeside       the TMA kernel, one CTA of 4 warps (6 stages each) per SM: a large render
//                 beside the leaf hash of the same merge (cm_ingest_render)
//   kBesideSmall  the register kernel, one 8-warp CTA per SM: a small render beside the leaf hash
// A launch group's work items are row chunks of render_item_bytes(w) bytes of one source
// plane; render_grid gives the launch's CTA count for `chunks` items. render_prepare() once
// per device before the first launch.
enum class RenderWidth { kFull, kHalf, kBeside, kBesideSmall };
cudaError_t launch_render(const RenderParams &p, int grid, RenderWidth w, cudaStream_t stream);
cudaError_t render_prepare();
uint32_t render_item_bytes(RenderWidth w);
int render_grid(uint64_t chunks, int num_sms, RenderWidth w);

// Bounds-checked builds: reads and zeroes the render kernels' violation count on the
// current device (0 in other builds).
cudaError_t take_render_bounds_violations(unsigned int *out);

}  // namespace cm
