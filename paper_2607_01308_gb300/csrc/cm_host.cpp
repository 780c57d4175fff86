// Host core of libcm: contexts, LatentFragmentSet state, canonical order and
// launch orchestration behind the C ABI of include/cm.h.
//
//   cm_fragment_id / cm_ingest   Id(C) and the norm key on the GPU, then the set
//                                insert on the host (Algorithm 2, Id / Ingest)
//   cm_union                     set union over 16-byte ids (Eq. setunion)
//   cm_render                    canonical order (Algorithm 1) on the host, then
//                                one fused copy-and-rotate launch (Eq. bagmerge-k/v)
//   cm_bagmerge                  the same launch in a caller-given order (Section 4.2)
#include "cm.h"
#include "cm_testing.h"

#include <algorithm>
#include <array>
#include <cmath>
#include <cstdio>
#include <cstddef>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <string>
#include <unordered_map>
#include <vector>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "cm_kernels.h"

namespace {

thread_local std::string g_last_error;

// NVTX range for the duration of a call (the library's phases in a profiler timeline).
struct TraceRange {
    explicit TraceRange(const char *name) { nvtxRangePushA(name); }
    ~TraceRange() { nvtxRangePop(); }
};

cm_status fail(cm_status st, const std::string &msg) {
    g_last_error = msg;
    return st;
}

cm_status cuda_fail(cudaError_t e, const char *what) {
    return fail(CM_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define CM_CUDA_TRY(expr, what)                              \
    do {                                                      \
        cudaError_t e_ = (expr);                              \
        if (e_ != cudaSuccess) return cuda_fail(e_, (what));  \
    } while (0)

// Makes `device` current for the scope of a call and restores the caller's device.
class DeviceScope {
  public:
    explicit DeviceScope(int device) {
        ok_ = cudaGetDevice(&prev_) == cudaSuccess;
        if (ok_ && prev_ != device) ok_ = cudaSetDevice(device) == cudaSuccess;
        changed_ = ok_ && prev_ != device;
    }
    ~DeviceScope() {
        if (changed_) cudaSetDevice(prev_);
    }
    bool ok() const { return ok_; }

  private:
    int prev_ = 0;
    bool ok_ = false;
    bool changed_ = false;
};

using IdKey = std::array<uint8_t, 16>;   // operator< is lexicographic = big-endian numeric

IdKey key_of(const cm_id &id) {
    IdKey k;
    std::memcpy(k.data(), id.b, 16);
    return k;
}

struct Record {
    cm_id id;
    int32_t L, H, T, d;
    const void *k;
    const void *v;
    std::vector<uint64_t> Q;   // routing-layer norm key Q[t]
};

bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cm_status validate_fragment(const cm_fragment *f) {
    if (!f) return fail(CM_ERR_INVALID_ARG, "fragment descriptor is NULL");
    if (f->num_layers < 1 || f->num_layers > 65535 || f->num_kv_heads < 1 ||
        f->num_kv_heads > 65535 || f->seq_len < 1)
        return fail(CM_ERR_INVALID_ARG, "fragment sizes out of range (layers and kv heads in "
                                        "[1, 65535], seq_len >= 1)");
    if (!is_pow2(f->head_dim) || f->head_dim < 16 || f->head_dim > 512)
        return fail(CM_ERR_INVALID_ARG, "head_dim must be a power of two in [16, 512]");
    if (!f->k || !f->v) return fail(CM_ERR_INVALID_ARG, "fragment k or v pointer is NULL");
    if (!aligned16(f->k) || !aligned16(f->v))
        return fail(CM_ERR_ALIGNMENT, "fragment k and v must be 16-byte aligned");
    const long double bytes = (long double)f->num_layers * f->num_kv_heads * f->seq_len *
                              f->head_dim * 2.0L * 2.0L;
    if (bytes > 9.0e15L) return fail(CM_ERR_UNSUPPORTED, "fragment too large");
    return CM_OK;
}

}  // namespace

// ------------------------------------------------------------------ context

struct cm_context {
    int device = 0;
    double theta = 1e6;
    int32_t routing_layer = -1;
    bool verify = false;
    int num_sms = 0;
    unsigned int *d_error = nullptr;   // set by a kernel whose bounded wait timed out
    std::mutex mu;
    // hashing scratch (device): leaf digests, inner levels, Q[t], compare flag
    uint8_t *d_scratch = nullptr;
    size_t scratch_bytes = 0;
    // pinned host staging for the root digest, Q[t] and the compare flag
    uint8_t *h_pinned = nullptr;
    void *h_pinned_dev = nullptr;   // its device-mapped address (null: use copy engines)
    size_t pinned_bytes = 0;
    int live_sets = 0;
    // kernel timing (cm_context_set_timing): events bracketing each launch
    bool timing = false;
    struct Pending {
        int kind;
        cudaEvent_t start, end;
        int kernels;   // kernels launched between the two events
    };
    std::vector<Pending> pending;
    std::vector<cudaEvent_t> event_pool;
    double time_ms[3] = {0, 0, 0};
    int64_t launches[3] = {0, 0, 0};
    int64_t leaf_fragments = 0;   // fragments hashed by the timed leaf-hash launches
    int64_t aux_launches = 0;     // readback and comparison launches while timing is on
    // RoPE frequencies theta^(-2j/d), j < d/2, for the last head_dim rendered
    std::vector<double> omega;
    int32_t omega_d = 0;
    // launch parameters of the render kernel (about 31 KB), reused by every launch
    std::unique_ptr<cm::RenderParams> render_params;
    int32_t render_warps = 16;   // warps per render CTA (cm_context_set_render_warps)
    bool dedup_bytes = false;    // re-delivery fast path (cm_context_set_dedup_by_bytes)
};

struct cm_set {
    cm_context *ctx = nullptr;
    bool has_shape = false;
    int32_t L = 0, H = 0, d = 0;
    std::map<IdKey, std::shared_ptr<const Record>> items;
};

namespace {

int32_t routing_layer_for(const cm_context *ctx, int32_t L) {
    return ctx->routing_layer < 0 ? L / 2 : ctx->routing_layer;
}

cm_status ensure_scratch(cm_context *ctx, size_t dev_bytes, size_t host_bytes) {
    if (dev_bytes > ctx->scratch_bytes) {
        const size_t old_dev = ctx->scratch_bytes;
        if (ctx->d_scratch) cudaFree(ctx->d_scratch);
        ctx->d_scratch = nullptr;
        ctx->scratch_bytes = 0;
        // grown by at least half its size, so a stream of slowly growing requests
        // reallocates (a device-wide synchronisation) only O(log) times
        const size_t want = std::max({dev_bytes, old_dev + old_dev / 2, (size_t)1 << 20});
        cudaError_t e = cudaMalloc(&ctx->d_scratch, want);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(CM_ERR_OOM, std::string("device scratch allocation failed: ") +
                                        cudaGetErrorString(e));
        }
        ctx->scratch_bytes = want;
    }
    if (host_bytes > ctx->pinned_bytes) {
        const size_t old_host = ctx->pinned_bytes;
        if (ctx->h_pinned) cudaFreeHost(ctx->h_pinned);
        ctx->h_pinned = nullptr;
        ctx->h_pinned_dev = nullptr;
        ctx->pinned_bytes = 0;
        const size_t want = std::max({host_bytes, old_host + old_host / 2, (size_t)1 << 16});
        cudaError_t e = cudaHostAlloc(reinterpret_cast<void **>(&ctx->h_pinned), want,
                                      cudaHostAllocMapped);
        if (e != cudaSuccess) {                    // no mapped host memory: a plain one
            cudaGetLastError();
            e = cudaHostAlloc(reinterpret_cast<void **>(&ctx->h_pinned), want, cudaHostAllocDefault);
        }
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(CM_ERR_OOM, std::string("pinned host allocation failed: ") +
                                        cudaGetErrorString(e));
        }
        // small results are written there by the SMs (readback.cu) when it is mapped
        if (cudaHostGetDevicePointer(&ctx->h_pinned_dev, ctx->h_pinned, 0) != cudaSuccess) {
            cudaGetLastError();
            ctx->h_pinned_dev = nullptr;
        }
        ctx->pinned_bytes = want;
    }
    return CM_OK;
}

// Reads a small device result (`bytes` at `src`) into ctx->h_pinned, enqueued on
// `stream`: stored by the SMs through the buffer's mapped address when both are 4-byte
// granular (so the read does not wait behind bulk device-to-host copies of other
// streams on the copy engine), else by a copy.
cudaError_t read_small(cm_context *ctx, const void *src, size_t bytes, cudaStream_t stream) {
    if (ctx->h_pinned_dev && bytes % 4 == 0 && (reinterpret_cast<uintptr_t>(src) & 3u) == 0) {
        if (ctx->timing) ++ctx->aux_launches;
        return cm::launch_readback(ctx->h_pinned_dev, src, bytes, stream);
    }
    return cudaMemcpyAsync(ctx->h_pinned, src, bytes, cudaMemcpyDeviceToHost, stream);
}

// BLAKE2s parameter block (32 bytes) of the tree, node offset and depth zero,
// xored into the IV: digest 16, no key, fanout 16, depth 255 (unlimited),
// leaf 1024, inner 16, salt = <L, H, d, 1 (bf16)> as little-endian uint16,
// personalisation = <T> as a little-endian uint64.
cm::TreeParams tree_params(int32_t L, int32_t H, int32_t d, int32_t T) {
    static const uint32_t iv[8] = {0x6A09E667u, 0xBB67AE85u, 0x3C6EF372u, 0xA54FF53Au,
                                   0x510E527Fu, 0x9B05688Cu, 0x1F83D9ABu, 0x5BE0CD19u};
    uint8_t p[32];
    std::memset(p, 0, sizeof p);
    p[0] = cm::kDigestBytes;
    p[1] = 0;
    p[2] = cm::kFanout;
    p[3] = 255;
    const uint32_t leaf = cm::kLeafBytes;
    for (int i = 0; i < 4; ++i) p[4 + i] = (uint8_t)(leaf >> (8 * i));
    p[15] = cm::kDigestBytes;   // inner length
    const uint16_t salt[4] = {(uint16_t)L, (uint16_t)H, (uint16_t)d, 1};
    for (int i = 0; i < 4; ++i) {
        p[16 + 2 * i] = (uint8_t)(salt[i] & 0xFF);
        p[17 + 2 * i] = (uint8_t)(salt[i] >> 8);
    }
    const uint64_t person = (uint64_t)T;
    for (int i = 0; i < 8; ++i) p[24 + i] = (uint8_t)(person >> (8 * i));
    cm::TreeParams tp;
    for (int i = 0; i < 8; ++i) {
        const uint32_t w = (uint32_t)p[4 * i] | ((uint32_t)p[4 * i + 1] << 8) |
                           ((uint32_t)p[4 * i + 2] << 16) | ((uint32_t)p[4 * i + 3] << 24);
        tp.h_base[i] = iv[i] ^ w;
    }
    return tp;
}

uint64_t ceil_div(uint64_t a, uint64_t b) { return (a + b - 1) / b; }

enum { kTimeLeaf = 0, kTimeInner = 1, kTimeRender = 2 };

cudaEvent_t take_event(cm_context *ctx) {
    if (!ctx->event_pool.empty()) {
        cudaEvent_t e = ctx->event_pool.back();
        ctx->event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return e;
}

// Runs `launch` (which launches `kernels` kernels) on `stream`; when timing is on,
// brackets it with two events.
template <class F>
cudaError_t timed_launch(cm_context *ctx, int kind, cudaStream_t stream, F &&launch,
                         int kernels = 1) {
    if (!ctx->timing) return launch();
    cudaEvent_t a = take_event(ctx), b = take_event(ctx);
    if (!a || !b) return launch();
    cudaEventRecord(a, stream);
    const cudaError_t e = launch();
    cudaEventRecord(b, stream);
    ctx->pending.push_back({kind, a, b, kernels});
    return e;
}

// Id(C) and Q[t] of n fragments in one pass: the leaf-hash launches of all
// fragments (with their norm keys), then the tree levels above the leaves (level 1,
// then the levels above it: two launches per kMaxGroup fragments), then a single copy
// of every root digest and norm key to the host and one synchronisation. Caller holds ctx->mu and the device scope.
//   device scratch: [roots n x 16][Q of fragment 0]...[Q of fragment n-1][levels...]
cm_status fragments_digest(cm_context *ctx, const cm_fragment *const *frags, size_t n,
                           cudaStream_t stream, cm_id *ids, std::vector<uint64_t> *Qs) {
    struct Layout {
        std::vector<uint64_t> sizes;
        std::vector<size_t> level_off;
        size_t q_off;
        uint64_t plane, stream_bytes;
        int32_t rl;
        cm::TreeParams tp;
    };
    std::vector<Layout> lay(n);
    const size_t roots_bytes = n * 16;
    size_t off = roots_bytes;
    for (size_t i = 0; i < n; ++i) {
        const cm_fragment *f = frags[i];
        Layout &l = lay[i];
        l.rl = routing_layer_for(ctx, f->num_layers);
        if (l.rl >= f->num_layers) return fail(CM_ERR_INVALID_ARG, "routing layer >= num_layers");
        l.plane = (uint64_t)f->num_kv_heads * f->seq_len * f->head_dim * 2;
        l.stream_bytes = 2ull * f->num_layers * l.plane;
        l.sizes.assign(1, ceil_div(l.stream_bytes, cm::kLeafBytes));
        while (l.sizes.size() == 1 || l.sizes.back() > 1)
            l.sizes.push_back(ceil_div(l.sizes.back(), cm::kFanout));
        l.q_off = off;
        off += (size_t)f->seq_len * 8;
        l.tp = tree_params(f->num_layers, f->num_kv_heads, f->head_dim, f->seq_len);
    }
    const size_t host_bytes = off;     // roots and norm keys, copied back in one piece
    // arrival counters of every node at levels >= 2 follow the norm keys, so that one
    // memset zeroes both before the launches
    std::vector<size_t> arr_off(n);
    for (size_t i = 0; i < n; ++i) {
        arr_off[i] = off;
        for (size_t k = 2; k < lay[i].sizes.size(); ++k) off += (size_t)lay[i].sizes[k] * 4;
    }
    const size_t zero_end = off;
    off = (off + 255) & ~(size_t)255;
    for (size_t i = 0; i < n; ++i) {
        Layout &l = lay[i];
        if (l.sizes.size() > (size_t)cm::kMaxLevels)
            return fail(CM_ERR_UNSUPPORTED, "fragment too large for the hash tree depth");
        for (size_t k = 0; k + 1 < l.sizes.size(); ++k) {   // the root goes to the roots area
            l.level_off.push_back(off);
            off += ((size_t)l.sizes[k] * cm::kDigestBytes + 255) & ~(size_t)255;
        }
    }
    cm_status st = ensure_scratch(ctx, off, host_bytes);
    if (st != CM_OK) return st;
    uint8_t *base = ctx->d_scratch;

    CM_CUDA_TRY(cudaMemsetAsync(base + roots_bytes, 0, zero_end - roots_bytes, stream),
                "zeroing the norm keys and arrival counters");
    // level 0 of up to kMaxLeafGroup fragments per launch
    std::unique_ptr<cm::LeafGroup> grp(new cm::LeafGroup);
    for (size_t g0 = 0; g0 < n; g0 += (size_t)cm::kMaxLeafGroup) {
        const size_t gn = std::min(n - g0, (size_t)cm::kMaxLeafGroup);
        std::memset(grp.get(), 0, sizeof(cm::LeafGroup));
        grp->count = (uint32_t)gn;
        for (size_t q = 0; q < gn; ++q) {
            const cm_fragment *f = frags[g0 + q];
            const Layout &l = lay[g0 + q];
            cm::LeafLaunch &a = grp->frag[q];
            a.k = static_cast<const uint8_t *>(f->k);
            a.v = static_cast<const uint8_t *>(f->v);
            a.plane_bytes = l.plane;
            a.stream_bytes = l.stream_bytes;
            a.num_leaves = l.sizes[0];
            a.norm_begin = 2ull * (uint64_t)l.rl * l.plane;
            a.row_bytes = (uint32_t)f->head_dim * 2;
            a.seq_len = (uint32_t)f->seq_len;
            a.norm_key = reinterpret_cast<unsigned long long *>(base + l.q_off);
            a.digests = base + l.level_off[0];
            a.tree = l.tp;
            grp->block_begin[q + 1] = grp->block_begin[q] + ceil_div(a.num_leaves, (uint64_t)cm::kLeafBlockThreads);
        }
        if (grp->block_begin[gn] > 0x7FFFFFFFull)
            return fail(CM_ERR_UNSUPPORTED, "leaf-hash launch exceeds 2^31 - 1 blocks");
        CM_CUDA_TRY(timed_launch(ctx, kTimeLeaf, stream,
                                 [&] { return cm::launch_leaf_hash_group(*grp, stream); }),
                    "leaf hash launch");
        if (ctx->timing) ctx->leaf_fragments += (int64_t)gn;
    }
    std::unique_ptr<cm::TreeTop> top(new cm::TreeTop);
    std::memset(top.get(), 0, sizeof(cm::TreeTop));
    auto flush = [&]() -> cudaError_t {
        if (top->count == 0) return cudaSuccess;
        const int kernels = cm::tree_top_kernels(*top);
        const cudaError_t e = timed_launch(
            ctx, kTimeInner, stream, [&] { return cm::launch_tree_top(*top, stream); }, kernels);
        std::memset(top.get(), 0, sizeof(cm::TreeTop));
        return e;
    };
    for (size_t i = 0; i < n; ++i) {
        const Layout &l = lay[i];
        const uint32_t c = top->count;
        cm::TreeTopFragment &tf = top->frag[c];
        tf.levels = (uint32_t)l.sizes.size();
        size_t a_off = arr_off[i];
        for (size_t k = 0; k < l.sizes.size(); ++k) {
            tf.size[k] = l.sizes[k];
            tf.level[k] = (k + 1 == l.sizes.size()) ? base + 16 * i : base + l.level_off[k];
            if (k >= 2) {
                tf.arrivals[k] = reinterpret_cast<uint32_t *>(base + a_off);
                a_off += (size_t)l.sizes[k] * 4;
            }
        }
        tf.tree = l.tp;
        top->node_begin[c + 1] = top->node_begin[c] + l.sizes[1];
        top->count = c + 1;
        if (top->count == (uint32_t)cm::kMaxGroup) CM_CUDA_TRY(flush(), "tree-top launch");
    }
    CM_CUDA_TRY(flush(), "tree-top launch");
    CM_CUDA_TRY(read_small(ctx, base, host_bytes, stream),
                "digest copy");
    CM_CUDA_TRY(cudaStreamSynchronize(stream), "ingest synchronisation");
    for (size_t i = 0; i < n; ++i) {
        std::memcpy(ids[i].b, ctx->h_pinned + 16 * i, 16);
        if (Qs) {
            Qs[i].resize((size_t)frags[i]->seq_len);
            std::memcpy(Qs[i].data(), ctx->h_pinned + lay[i].q_off, (size_t)frags[i]->seq_len * 8);
        }
    }
    return CM_OK;
}

// Reads and clears the context's error word on `stream` (synchronising it).
cm_status take_device_error(cm_context *ctx, cudaStream_t stream) {
    cm_status st = ensure_scratch(ctx, 0, 16);
    if (st != CM_OK) return st;
    CM_CUDA_TRY(read_small(ctx, ctx->d_error, sizeof(unsigned int), stream),
                "error word copy");
    CM_CUDA_TRY(cudaStreamSynchronize(stream), "error word synchronisation");
    unsigned int e;
    std::memcpy(&e, ctx->h_pinned, sizeof e);
    if (e == 0) return CM_OK;
    CM_CUDA_TRY(cudaMemsetAsync(ctx->d_error, 0, sizeof(unsigned int), stream), "error word reset");
    CM_CUDA_TRY(cudaStreamSynchronize(stream), "error word synchronisation");
    return fail(CM_ERR_TIMEOUT, "a bounded wait inside a render kernel timed out; that render's "
                                "output is incomplete");
}

// Byte comparison of a new fragment against a stored record with the same id.
cm_status bytes_equal(cm_context *ctx, const cm_fragment *f, const Record &r, cudaStream_t stream,
                      bool *equal) {
    const uint64_t bytes = (uint64_t)f->num_layers * f->num_kv_heads * f->seq_len * f->head_dim * 2;
    if (r.L != f->num_layers || r.H != f->num_kv_heads || r.T != f->seq_len || r.d != f->head_dim) {
        *equal = false;
        return CM_OK;
    }
    cm_status st = ensure_scratch(ctx, 256, 16);
    if (st != CM_OK) return st;
    auto *flag = reinterpret_cast<unsigned int *>(ctx->d_scratch);
    CM_CUDA_TRY(cudaMemsetAsync(flag, 0, sizeof(unsigned int), stream), "flag reset");
    CM_CUDA_TRY(cm::launch_compare(f->k, r.k, bytes, flag, stream), "compare launch");
    CM_CUDA_TRY(cm::launch_compare(f->v, r.v, bytes, flag, stream), "compare launch");
    CM_CUDA_TRY(read_small(ctx, flag, sizeof(unsigned int), stream),
                "flag copy");
    CM_CUDA_TRY(cudaStreamSynchronize(stream), "compare synchronisation");
    unsigned int h;
    std::memcpy(&h, ctx->h_pinned, sizeof h);
    *equal = h == 0;
    return CM_OK;
}

// One slot of a render: a fragment, its output offset and its set's contiguous
// output (ignored for paged outputs).
struct Slot {
    const void *k;
    const void *v;
    int64_t T;
    int64_t offset;
    void *k_out;
    void *v_out;
    int64_t capacity;
};

// Fused copy-and-rotate of slots already in order (offsets set), in launch groups
// of at most kMaxSlots slots and kMaxTablePairs (cos, sin) pairs. The slots may
// belong to several sets of one shape: each slot carries its own output.
cm_status launch_slots(cm_context *ctx, const std::vector<Slot> &slots, int32_t L, int32_t H,
                       int32_t d, cudaStream_t stream, uint32_t withhold_warp = 0,
                       const cm_paged_cache *paged = nullptr) {
    // the failure-injection hook withholds a TMA copy, so it runs the half-SM kernel (the
    // only one that waits)
    const int warps = withhold_warp ? 8 : ctx->render_warps;
    const int rows_per_chunk = (int)cm::render_item_bytes(warps) / (2 * d);
    const int half = d / 2;
    const int max_group = std::min<int>(cm::kMaxSlots, cm::kMaxTablePairs / half);
    const uint64_t planes = 2ull * L * H;
    int log2_pairs = 0;
    while ((1 << log2_pairs) < d / 16) ++log2_pairs;
    if (ctx->omega_d != d) {
        ctx->omega.resize((size_t)half);
        for (int j = 0; j < half; ++j) ctx->omega[(size_t)j] = std::pow(ctx->theta, -(2.0 * j) / d);
        ctx->omega_d = d;
    }
    if (!ctx->render_params) ctx->render_params.reset(new cm::RenderParams);
    cm::RenderParams *p = ctx->render_params.get();
    for (size_t g0 = 0; g0 < slots.size(); g0 += (size_t)max_group) {
        const size_t n = std::min(slots.size() - g0, (size_t)max_group);
        // the kernel reads the header, slot[0, n) and the (cos, sin) pairs of those slots
        // that rotate, all written below; the rest of the block keeps older values
        std::memset(p, 0, offsetof(cm::RenderParams, slot));
        std::memset(p->slot, 0, n * sizeof(cm::RenderSlot));
        p->num_layers = L;
        p->num_heads = H;
        p->head_dim = d;
        p->num_slots = (int32_t)n;
        p->rows_per_chunk = rows_per_chunk;
        p->log2_pairs_per_row = log2_pairs;
        uint64_t chunk = 0;
        for (size_t i = 0; i < n; ++i) {
            const Slot &s = slots[g0 + i];
            cm::RenderSlot &rs = p->slot[i];
            rs.k = s.k;
            rs.v = s.v;
            rs.k_out = s.k_out;
            rs.v_out = s.v_out;
            rs.capacity = s.capacity;
            rs.seq_len = s.T;
            rs.offset = s.offset;
            rs.rotate = s.offset != 0;
            rs.table_base = (int32_t)i * half;
            const uint64_t cpp = ceil_div((uint64_t)s.T, (uint64_t)rows_per_chunk);
            rs.chunk_begin = (uint32_t)chunk;
            rs.chunks_per_plane = (uint32_t)cpp;
            chunk += cpp * planes;
            // delta angle a_j = s * theta^(-2j/d) in fp64 (Section 4.2, Eq. bagmerge-k);
            // the slot at offset 0 is copied and needs no table
            if (rs.rotate) {
                for (int j = 0; j < half; ++j) {
                    const double a = (double)s.offset * ctx->omega[(size_t)j];
                    p->cs[2 * (i * half + j)] = std::cos(a);
                    p->cs[2 * (i * half + j) + 1] = std::sin(a);
                }
            }
        }
        if (chunk > 0xFFFFFFFFull)
            return fail(CM_ERR_UNSUPPORTED, "render launch group exceeds 2^32 work items");
        p->total_chunks = (uint32_t)chunk;
        p->error = ctx->d_error;
        p->withhold_warp = g0 == 0 ? withhold_warp : 0;
        if (paged) {
            p->paged = 1;
            p->k_pool = paged->k_pool;
            p->v_pool = paged->v_pool;
            p->block_table = paged->block_table;
            p->table_entries = paged->table_entries;
            p->block_size = paged->block_size;
            p->log2_block_size = is_pow2(paged->block_size)
                                     ? (int32_t)__builtin_ctzll((unsigned long long)paged->block_size)
                                     : -1;
            p->stride_block = paged->stride_block;
            p->stride_layer = paged->stride_layer;
            p->stride_head = paged->stride_head;
            p->stride_token = paged->stride_token;
        }
        const int grid = cm::render_grid(chunk, ctx->num_sms, warps);
        CM_CUDA_TRY(timed_launch(ctx, kTimeRender, stream,
                                 [&] { return cm::launch_render(*p, grid, warps, stream); }),
                    "render launch");
    }
    return CM_OK;
}

cm_status validate_outputs(void *k_out, void *v_out, int64_t capacity, int64_t total) {
    if (capacity < total)
        return fail(CM_ERR_CAPACITY, "rendered length " + std::to_string(total) +
                                         " exceeds capacity_tokens " + std::to_string(capacity));
    if (total == 0) return CM_OK;
    if (!k_out || !v_out) return fail(CM_ERR_INVALID_ARG, "k_out or v_out is NULL");
    if (!aligned16(k_out) || !aligned16(v_out))
        return fail(CM_ERR_ALIGNMENT, "k_out and v_out must be 16-byte aligned");
    return CM_OK;
}

// Canonical order of Algorithm 1: descending tail sum of the norm key over the
// last T* = min T positions (the integer form of rho, Eq. rho), ties by
// descending id read big-endian.
std::vector<std::shared_ptr<const Record>> canonical_order(const cm_set *set) {
    std::vector<std::shared_ptr<const Record>> recs;
    recs.reserve(set->items.size());
    int64_t t_star = INT64_MAX;
    for (const auto &kv : set->items) {
        recs.push_back(kv.second);
        t_star = std::min<int64_t>(t_star, kv.second->T);
    }
    struct Keyed {
        unsigned __int128 S;
        IdKey id;
        std::shared_ptr<const Record> r;
    };
    std::vector<Keyed> keyed;
    keyed.reserve(recs.size());
    for (auto &r : recs) {
        // each Q[t] is at most H (2^44 - 1): when H T* (2^44 - 1) < 2^64 the tail sum
        // cannot wrap in 64 bits, and a plain 64-bit sum (which vectorises) is exact
        const uint64_t *q = r->Q.data() + (r->T - t_star);
        unsigned __int128 S = 0;
        if ((unsigned __int128)r->H * (uint64_t)t_star * ((1ull << 44) - 1) <
            ((unsigned __int128)1 << 64)) {
            uint64_t s64 = 0;
            for (int64_t t = 0; t < t_star; ++t) s64 += q[t];
            S = s64;
        } else {
            for (int64_t t = 0; t < t_star; ++t) S += q[t];
        }
        keyed.push_back({S, key_of(r->id), r});
    }
    std::sort(keyed.begin(), keyed.end(), [](const Keyed &a, const Keyed &b) {
        if (a.S != b.S) return a.S > b.S;
        return a.id > b.id;
    });
    std::vector<std::shared_ptr<const Record>> out;
    out.reserve(keyed.size());
    for (auto &k : keyed) out.push_back(k.r);
    return out;
}

template <class F>
cm_status guarded(F &&f) {
    try {
        return f();
    } catch (const std::bad_alloc &) {
        return fail(CM_ERR_OOM, "host allocation failed");
    } catch (...) {
        return fail(CM_ERR_INVALID_ARG, "unexpected internal error");
    }
}

// Re-delivery fast path: the deliveries of one ingest call that are byte-identical to
// a fragment their set already holds or to an earlier delivery of the call. A
// delivery is compared with at most kMaxCandidates fragments of its shape and length
// (the set's records first, then the call's earlier deliveries, the latest first):
// their first 4 KiB in one pass, then all bytes of the first candidate whose prefix
// matched; identical (k, v) pointers count as equal without a comparison. Results:
// rec[i] is the equal record, else from[i] the equal earlier delivery, else neither
// (hash it).
constexpr int kMaxCandidates = 16;

cm_status find_redeliveries(cm_context *ctx, cm_set *const *sets,
                            const std::vector<const cm_fragment *> &fp, cudaStream_t stream,
                            std::vector<std::shared_ptr<const Record>> &rec,
                            std::vector<int32_t> &from) {
    const size_t n = fp.size();
    rec.assign(n, nullptr);
    from.assign(n, -1);
    struct Cand {
        size_t delivery;
        std::shared_ptr<const Record> r;   // a record, or null for delivery `other`
        size_t other;
    };
    std::vector<Cand> cands;
    auto same_shape = [](const cm_fragment *f, int32_t L, int32_t H, int32_t T, int32_t d) {
        return f->num_layers == L && f->num_kv_heads == H && f->seq_len == T && f->head_dim == d;
    };
    for (size_t i = 0; i < n; ++i) {
        const cm_fragment *f = fp[i];
        int found = 0;
        bool same_buffers = false;
        for (const auto &kv : sets[i]->items) {
            const Record &r = *kv.second;
            if (!same_shape(f, r.L, r.H, r.T, r.d)) continue;
            if (r.k == f->k && r.v == f->v) {
                rec[i] = kv.second;
                same_buffers = true;
                break;
            }
            if (found < kMaxCandidates) {
                cands.push_back({i, kv.second, 0});
                ++found;
            }
        }
        for (size_t j = i; j-- > 0 && !same_buffers;) {
            const cm_fragment *g = fp[j];
            if (!same_shape(f, g->num_layers, g->num_kv_heads, g->seq_len, g->head_dim)) continue;
            if (g->k == f->k && g->v == f->v) {
                from[i] = (int32_t)j;
                same_buffers = true;
                break;
            }
            if (found < kMaxCandidates) {
                cands.push_back({i, nullptr, j});
                ++found;
            }
        }
        if (same_buffers)
            while (!cands.empty() && cands.back().delivery == i) cands.pop_back();
    }
    if (cands.empty()) return CM_OK;
    // one comparison pass over a list of candidate pairs: differ[c] = 1 if pair c differs
    // (its first 4 KiB of K only, or all of it)
    auto compare = [&](const std::vector<size_t> &which, bool full,
                       std::vector<uint32_t> &differ) -> cm_status {
        differ.assign(which.size(), 1u);
        cm_status st = ensure_scratch(ctx, which.size() * 4, which.size() * 4);
        if (st != CM_OK) return st;
        auto *d_differ = reinterpret_cast<uint32_t *>(ctx->d_scratch);
        CM_CUDA_TRY(cudaMemsetAsync(d_differ, 0, which.size() * 4, stream), "comparison flags reset");
        for (size_t c0 = 0; c0 < which.size(); c0 += (size_t)cm::kMaxComparePairs) {
            cm::CompareLaunch cl;
            std::memset(&cl, 0, sizeof cl);
            const size_t cn = std::min(which.size() - c0, (size_t)cm::kMaxComparePairs);
            for (size_t q = 0; q < cn; ++q) {
                const Cand &c = cands[which[c0 + q]];
                const cm_fragment *f = fp[c.delivery];
                const void *bk = c.r ? c.r->k : fp[c.other]->k;
                const void *bv = c.r ? c.r->v : fp[c.other]->v;
                const uint64_t vecs =
                    (uint64_t)f->num_layers * f->num_kv_heads * f->seq_len * f->head_dim * 2 / 16;
                cl.pair[q] = {static_cast<const uint4 *>(f->k), static_cast<const uint4 *>(f->v),
                              static_cast<const uint4 *>(bk), static_cast<const uint4 *>(bv), vecs};
                cl.chunk_begin[q + 1] =
                    cl.chunk_begin[q] + 2 * ceil_div(vecs, (uint64_t)cm::kCompareChunkVecs);
            }
            cl.count = (uint32_t)cn;
            cl.differ = d_differ + c0;
            CM_CUDA_TRY(full ? cm::launch_compare_full(cl, ctx->num_sms, stream)
                             : cm::launch_compare_prefix(cl, stream),
                        "comparison launch");
            if (ctx->timing) ++ctx->aux_launches;
        }
        CM_CUDA_TRY(read_small(ctx, d_differ, which.size() * 4, stream),
                    "comparison flags copy");
        CM_CUDA_TRY(cudaStreamSynchronize(stream), "comparison synchronisation");
        std::memcpy(differ.data(), ctx->h_pinned, which.size() * 4);
        return CM_OK;
    };
    // first the 4 KiB prefixes of every pair, then the whole of one pair per delivery:
    // its first candidate whose prefix matched (one full comparison suffices, and
    // re-deliveries of one fragment would otherwise all be compared with each other)
    std::vector<size_t> all(cands.size());
    for (size_t c = 0; c < cands.size(); ++c) all[c] = c;
    std::vector<uint32_t> prefix_differ, full_differ;
    cm_status st = compare(all, false, prefix_differ);
    if (st != CM_OK) return st;
    std::vector<size_t> chosen;
    std::vector<bool> has_choice(n, false);
    for (size_t c = 0; c < cands.size(); ++c) {
        const size_t i = cands[c].delivery;
        if (prefix_differ[c] != 0 || has_choice[i]) continue;
        has_choice[i] = true;
        chosen.push_back(c);
    }
    if (chosen.empty()) return CM_OK;
    st = compare(chosen, true, full_differ);
    if (st != CM_OK) return st;
    for (size_t q = 0; q < chosen.size(); ++q) {
        if (full_differ[q] != 0) continue;
        const Cand &c = cands[chosen[q]];
        if (c.r)
            rec[c.delivery] = c.r;
        else
            from[c.delivery] = (int32_t)c.other;
    }
    return CM_OK;
}

// Ingest (Algorithm 2) of n deliveries, delivery i into sets[i] (several entries
// may name one set): one GPU pass for all of them, then the insertions in delivery
// order, so a delivery whose id its set already holds (before the batch or from an
// earlier delivery of it) is absorbed. Nothing is inserted if validation fails.
cm_status ingest_deliveries(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                            cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed) {
    if (n == 0) return CM_OK;
    cm_context *ctx = sets[0]->ctx;
    struct Shape {
        bool has;
        int32_t L, H, d;
    };
    std::unordered_map<const cm_set *, Shape> shape;
    std::vector<const cm_fragment *> fp((size_t)n);
    for (int32_t i = 0; i < n; ++i) {
        const cm_set *set = sets[i];
        if (set->ctx != ctx) return fail(CM_ERR_INVALID_ARG, "sets belong to different contexts");
        const cm_fragment *f = &frags[i];
        cm_status st = validate_fragment(f);
        if (st != CM_OK) return st;
        auto it = shape.find(set);
        if (it == shape.end())
            it = shape.emplace(set, Shape{set->has_shape, set->L, set->H, set->d}).first;
        Shape &sh = it->second;
        if (!sh.has) {
            sh = Shape{true, f->num_layers, f->num_kv_heads, f->head_dim};
        } else if (f->num_layers != sh.L || f->num_kv_heads != sh.H || f->head_dim != sh.d) {
            return fail(CM_ERR_SHAPE_MISMATCH,
                        "fragment (layers, kv_heads, head_dim) differ from the set's");
        }
        if (routing_layer_for(ctx, f->num_layers) >= f->num_layers)
            return fail(CM_ERR_INVALID_ARG, "routing layer >= num_layers");
        fp[(size_t)i] = f;
    }
    std::lock_guard<std::mutex> lock(ctx->mu);
    DeviceScope scope(ctx->device);
    if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
    const cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
    // with the re-delivery fast path on, deliveries byte-identical to a known fragment
    // take its id and norm key and are not hashed
    std::vector<std::shared_ptr<const Record>> same_rec;
    std::vector<int32_t> same_as;
    cm_status st = CM_OK;
    if (ctx->dedup_bytes) {
        st = find_redeliveries(ctx, sets, fp, cs, same_rec, same_as);
        if (st != CM_OK) return st;
    } else {
        same_rec.assign((size_t)n, nullptr);
        same_as.assign((size_t)n, -1);
    }
    std::vector<const cm_fragment *> to_hash;
    std::vector<size_t> hashed_as((size_t)n, 0);
    for (int32_t i = 0; i < n; ++i)
        if (!same_rec[(size_t)i] && same_as[(size_t)i] < 0) {
            hashed_as[(size_t)i] = to_hash.size();
            to_hash.push_back(fp[(size_t)i]);
        }
    std::vector<cm_id> hashed_ids(to_hash.size());
    std::vector<std::vector<uint64_t>> hashed_Q(to_hash.size());
    if (!to_hash.empty()) {
        st = fragments_digest(ctx, to_hash.data(), to_hash.size(), cs, hashed_ids.data(),
                              hashed_Q.data());
        if (st != CM_OK) return st;
    }
    // ids in delivery order; Qsrc[i] is where delivery i's norm key lives once delivery i
    // has been processed (its own record, a record it matched, or a hashed result)
    std::vector<cm_id> ids((size_t)n);
    std::vector<const std::vector<uint64_t> *> Qsrc((size_t)n, nullptr);
    for (int32_t i = 0; i < n; ++i) {
        cm_set *set = sets[i];
        const cm_fragment *f = fp[(size_t)i];
        std::vector<uint64_t> *own = nullptr;
        if (same_rec[(size_t)i]) {
            ids[(size_t)i] = same_rec[(size_t)i]->id;
            Qsrc[(size_t)i] = &same_rec[(size_t)i]->Q;
        } else if (same_as[(size_t)i] >= 0) {
            ids[(size_t)i] = ids[(size_t)same_as[(size_t)i]];
            Qsrc[(size_t)i] = Qsrc[(size_t)same_as[(size_t)i]];
        } else {
            ids[(size_t)i] = hashed_ids[hashed_as[(size_t)i]];
            own = &hashed_Q[hashed_as[(size_t)i]];
            Qsrc[(size_t)i] = own;
        }
        if (out_ids) out_ids[i] = ids[(size_t)i];
        const IdKey key = key_of(ids[(size_t)i]);
        auto it = set->items.find(key);
        if (it != set->items.end()) {
            // a byte match against this very record needs no second look at the bytes
            if (ctx->verify && same_rec[(size_t)i] != it->second) {
                bool equal = false;
                st = bytes_equal(ctx, f, *it->second, cs, &equal);
                if (st != CM_OK) return st;
                if (!equal) return fail(CM_ERR_COLLISION, "content address hit with different bytes");
            }
            if (out_absorbed) out_absorbed[i] = 1;
            continue;
        }
        auto rec = std::make_shared<Record>();
        rec->id = ids[(size_t)i];
        rec->L = f->num_layers;
        rec->H = f->num_kv_heads;
        rec->T = f->seq_len;
        rec->d = f->head_dim;
        rec->k = f->k;
        rec->v = f->v;
        if (own)
            rec->Q = std::move(*own);
        else
            rec->Q = *Qsrc[(size_t)i];
        Qsrc[(size_t)i] = &rec->Q;
        set->items.emplace(key, std::move(rec));
        if (!set->has_shape) {
            set->has_shape = true;
            set->L = f->num_layers;
            set->H = f->num_kv_heads;
            set->d = f->head_dim;
        }
        if (out_absorbed) out_absorbed[i] = 0;
    }
    return CM_OK;
}

}  // namespace

extern "C" {

int32_t cm_abi_version(void) { return CM_ABI_VERSION; }

const char *cm_status_string(cm_status s) {
    switch (s) {
        case CM_OK: return "CM_OK";
        case CM_ERR_INVALID_ARG: return "CM_ERR_INVALID_ARG";
        case CM_ERR_SHAPE_MISMATCH: return "CM_ERR_SHAPE_MISMATCH";
        case CM_ERR_CAPACITY: return "CM_ERR_CAPACITY";
        case CM_ERR_ALIGNMENT: return "CM_ERR_ALIGNMENT";
        case CM_ERR_COLLISION: return "CM_ERR_COLLISION";
        case CM_ERR_CUDA: return "CM_ERR_CUDA";
        case CM_ERR_OOM: return "CM_ERR_OOM";
        case CM_ERR_TIMEOUT: return "CM_ERR_TIMEOUT";
        case CM_ERR_UNSUPPORTED: return "CM_ERR_UNSUPPORTED";
    }
    return "CM_ERR_UNKNOWN";
}

const char *cm_last_error_message(void) { return g_last_error.c_str(); }

cm_status cm_context_create(int32_t device, double rope_theta, int32_t routing_layer,
                            int32_t verify_bytes_on_hit, cm_context **out) {
    return guarded([&]() -> cm_status {
        if (!out) return fail(CM_ERR_INVALID_ARG, "out is NULL");
        *out = nullptr;
        if (device < 0) return fail(CM_ERR_INVALID_ARG, "device must be >= 0");
        if (!(rope_theta > 0.0) || !std::isfinite(rope_theta))
            return fail(CM_ERR_INVALID_ARG, "rope_theta must be finite and > 0");
        int count = 0;
        CM_CUDA_TRY(cudaGetDeviceCount(&count), "cudaGetDeviceCount");
        if (device >= count) return fail(CM_ERR_INVALID_ARG, "no such CUDA device");
        DeviceScope scope(device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        std::unique_ptr<cm_context> ctx(new cm_context);
        ctx->device = device;
        ctx->theta = rope_theta;
        ctx->routing_layer = routing_layer;
        ctx->verify = verify_bytes_on_hit != 0;
        CM_CUDA_TRY(cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, device),
                    "multiprocessor count");
        CM_CUDA_TRY(cm::render_prepare(), "render kernel attributes");
        CM_CUDA_TRY(cudaMalloc(&ctx->d_error, sizeof(unsigned int)), "error word allocation");
        CM_CUDA_TRY(cudaMemset(ctx->d_error, 0, sizeof(unsigned int)), "error word reset");
        *out = ctx.release();
        return CM_OK;
    });
}

cm_status cm_context_destroy(cm_context *ctx) {
    if (!ctx) return CM_OK;
    return guarded([&]() -> cm_status {
        if (ctx->live_sets != 0)
            return fail(CM_ERR_INVALID_ARG, "context still has live sets");
        DeviceScope scope(ctx->device);
        if (ctx->d_scratch) cudaFree(ctx->d_scratch);
        if (ctx->h_pinned) cudaFreeHost(ctx->h_pinned);
        if (ctx->d_error) cudaFree(ctx->d_error);
        for (const auto &pe : ctx->pending) {
            cudaEventDestroy(pe.start);
            cudaEventDestroy(pe.end);
        }
        for (cudaEvent_t e : ctx->event_pool) cudaEventDestroy(e);
        delete ctx;
        return CM_OK;
    });
}

cm_status cm_set_create(cm_context *ctx, cm_set **out) {
    return guarded([&]() -> cm_status {
        if (!out) return fail(CM_ERR_INVALID_ARG, "out is NULL");
        *out = nullptr;
        if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
        std::lock_guard<std::mutex> lock(ctx->mu);
        cm_set *s = new cm_set;
        s->ctx = ctx;
        ++ctx->live_sets;
        *out = s;
        return CM_OK;
    });
}

cm_status cm_set_destroy(cm_set *set) {
    if (!set) return CM_OK;
    return guarded([&]() -> cm_status {
        {
            std::lock_guard<std::mutex> lock(set->ctx->mu);
            --set->ctx->live_sets;
        }
        delete set;
        return CM_OK;
    });
}

cm_status cm_fragment_id(cm_context *ctx, const cm_fragment *frag, cm_stream_t stream,
                         cm_id *out_id, uint64_t *out_norm_key) {
    TraceRange trace("cm_fragment_id");
    return guarded([&]() -> cm_status {
        if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
        if (!out_id) return fail(CM_ERR_INVALID_ARG, "out_id is NULL");
        cm_status st = validate_fragment(frag);
        if (st != CM_OK) return st;
        if (routing_layer_for(ctx, frag->num_layers) >= frag->num_layers)
            return fail(CM_ERR_INVALID_ARG, "routing layer >= num_layers");
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        std::vector<uint64_t> Q[1];
        st = fragments_digest(ctx, &frag, 1, reinterpret_cast<cudaStream_t>(stream), out_id,
                              out_norm_key ? Q : nullptr);
        if (st != CM_OK) return st;
        if (out_norm_key) std::memcpy(out_norm_key, Q[0].data(), Q[0].size() * sizeof(uint64_t));
        return CM_OK;
    });
}

cm_status cm_ingest(cm_set *set, const cm_fragment *frag, cm_stream_t stream, cm_id *out_id,
                    int32_t *out_absorbed) {
    return cm_ingest_batch(set, frag, 1, stream, out_id, out_absorbed);
}

cm_status cm_ingest_batch(cm_set *set, const cm_fragment *frags, int32_t n, cm_stream_t stream,
                          cm_id *out_ids, int32_t *out_absorbed) {
    TraceRange trace("cm_ingest");
    return guarded([&]() -> cm_status {
        if (!set) return fail(CM_ERR_INVALID_ARG, "set is NULL");
        if (n < 0 || (n > 0 && !frags)) return fail(CM_ERR_INVALID_ARG, "need n >= 0 fragments");
        const std::vector<cm_set *> sets((size_t)n, set);
        return ingest_deliveries(sets.data(), frags, n, stream, out_ids, out_absorbed);
    });
}

cm_status cm_ingest_many(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                         cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed) {
    TraceRange trace("cm_ingest");
    return guarded([&]() -> cm_status {
        if (n < 0 || (n > 0 && (!frags || !sets)))
            return fail(CM_ERR_INVALID_ARG, "need n >= 0 fragments and their sets");
        for (int32_t i = 0; i < n; ++i)
            if (!sets[i]) return fail(CM_ERR_INVALID_ARG, "a set is NULL");
        return ingest_deliveries(sets, frags, n, stream, out_ids, out_absorbed);
    });
}


cm_status cm_context_set_dedup_by_bytes(cm_context *ctx, int32_t enable) {
    if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
    std::lock_guard<std::mutex> lock(ctx->mu);
    ctx->dedup_bytes = enable != 0;
    return CM_OK;
}

cm_status cm_context_set_render_warps(cm_context *ctx, int32_t warps) {
    if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
    if (warps != 8 && warps != 16) return fail(CM_ERR_INVALID_ARG, "render warps must be 8 or 16");
    std::lock_guard<std::mutex> lock(ctx->mu);
    ctx->render_warps = warps;
    return CM_OK;
}

cm_status cm_context_set_timing(cm_context *ctx, int32_t enable) {
    if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
    std::lock_guard<std::mutex> lock(ctx->mu);
    ctx->timing = enable != 0;
    return CM_OK;
}

cm_status cm_context_kernel_times(cm_context *ctx, cm_kernel_times *out, int32_t reset) {
    return guarded([&]() -> cm_status {
        if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        for (const auto &pe : ctx->pending) {
            float ms = 0.f;
            CM_CUDA_TRY(cudaEventSynchronize(pe.end), "timing event");
            CM_CUDA_TRY(cudaEventElapsedTime(&ms, pe.start, pe.end), "timing event");
            ctx->time_ms[pe.kind] += ms;
            ctx->launches[pe.kind] += pe.kernels;
            ctx->event_pool.push_back(pe.start);
            ctx->event_pool.push_back(pe.end);
        }
        ctx->pending.clear();
        if (out) {
            out->leaf_hash_ms = ctx->time_ms[kTimeLeaf];
            out->leaf_hash_launches = ctx->launches[kTimeLeaf];
            out->leaf_hash_fragments = ctx->leaf_fragments;
            out->aux_launches = ctx->aux_launches;
            out->inner_hash_ms = ctx->time_ms[kTimeInner];
            out->inner_hash_launches = ctx->launches[kTimeInner];
            out->render_ms = ctx->time_ms[kTimeRender];
            out->render_launches = ctx->launches[kTimeRender];
        }
        if (reset) {
            for (int k = 0; k < 3; ++k) {
                ctx->time_ms[k] = 0;
                ctx->launches[k] = 0;
            }
            ctx->leaf_fragments = 0;
            ctx->aux_launches = 0;
        }
        return CM_OK;
    });
}

cm_status cm_union(cm_set *dst, const cm_set *src) {
    TraceRange trace("cm_union");
    return guarded([&]() -> cm_status {
        if (!dst || !src) return fail(CM_ERR_INVALID_ARG, "set is NULL");
        if (dst == src) return CM_OK;
        if (dst->ctx != src->ctx)
            return fail(CM_ERR_INVALID_ARG, "sets belong to different contexts");
        if (dst->has_shape && src->has_shape &&
            (dst->L != src->L || dst->H != src->H || dst->d != src->d))
            return fail(CM_ERR_SHAPE_MISMATCH, "sets have different shapes");
        for (const auto &kv : src->items) dst->items.emplace(kv.first, kv.second);
        if (!dst->has_shape && src->has_shape) {
            dst->has_shape = true;
            dst->L = src->L;
            dst->H = src->H;
            dst->d = src->d;
        }
        return CM_OK;
    });
}

cm_status cm_set_size(const cm_set *set, int64_t *out) {
    if (!set || !out) return fail(CM_ERR_INVALID_ARG, "set or out is NULL");
    *out = (int64_t)set->items.size();
    return CM_OK;
}

cm_status cm_set_seq_len(const cm_set *set, int64_t *out) {
    if (!set || !out) return fail(CM_ERR_INVALID_ARG, "set or out is NULL");
    int64_t total = 0;
    for (const auto &kv : set->items) total += kv.second->T;
    *out = total;
    return CM_OK;
}

cm_status cm_set_ids(const cm_set *set, cm_id *out, int64_t capacity) {
    if (!set) return fail(CM_ERR_INVALID_ARG, "set is NULL");
    if (capacity > 0 && !out) return fail(CM_ERR_INVALID_ARG, "out is NULL");
    int64_t i = 0;
    for (const auto &kv : set->items) {
        if (i >= capacity) break;
        out[i++] = kv.second->id;
    }
    return CM_OK;
}

namespace {

cm_status render_set(const cm_set *set, void *k_out, void *v_out, int64_t capacity_tokens,
                     cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order,
                     uint32_t withhold_warp, const cm_id *prev_order = nullptr,
                     int64_t prev_n = 0, int64_t *out_reused_tokens = nullptr,
                     const cm_paged_cache *paged = nullptr) {
    TraceRange trace("cm_render");
    return guarded([&]() -> cm_status {
        if (!set) return fail(CM_ERR_INVALID_ARG, "set is NULL");
        if (capacity_tokens < 0) return fail(CM_ERR_INVALID_ARG, "capacity_tokens < 0");
        if (prev_n < 0 || (prev_n > 0 && !prev_order))
            return fail(CM_ERR_INVALID_ARG, "prev_order is NULL or prev_n < 0");
        int64_t total = 0;
        for (const auto &kv : set->items) total += kv.second->T;
        cm_status st = validate_outputs(k_out, v_out, capacity_tokens, total);
        if (st != CM_OK) return st;
        if (paged && total > 0) {
            if (!paged->block_table) return fail(CM_ERR_INVALID_ARG, "block_table is NULL");
            if (paged->block_size < 1) return fail(CM_ERR_INVALID_ARG, "block_size < 1");
            if (paged->stride_block % 8 || paged->stride_layer % 8 || paged->stride_head % 8 ||
                paged->stride_token % 8 || paged->stride_block < 0 || paged->stride_layer < 0 ||
                paged->stride_head < 0 || paged->stride_token < 0)
                return fail(CM_ERR_ALIGNMENT, "paged strides must be non-negative multiples of 8 elements");
            if (paged->stride_token < set->d)
                return fail(CM_ERR_INVALID_ARG, "stride_token is smaller than head_dim");
        }
        const auto order = canonical_order(set);
        if (out_seq_len) *out_seq_len = total;
        if (out_order)
            for (size_t i = 0; i < order.size(); ++i) out_order[i] = order[i]->id;
        // slots of the common prefix of the previous and the new canonical order keep
        // their offsets, so their bytes in the buffer are already the render's
        size_t keep = 0;
        while (keep < order.size() && (int64_t)keep < prev_n &&
               std::memcmp(order[keep]->id.b, prev_order[keep].b, 16) == 0)
            ++keep;
        std::vector<Slot> slots;
        slots.reserve(order.size());
        int64_t s = 0, reused = 0;
        for (size_t i = 0; i < order.size(); ++i) {
            if (i < keep)
                reused += order[i]->T;
            else
                slots.push_back({order[i]->k, order[i]->v, order[i]->T, s, k_out, v_out,
                                 capacity_tokens});
            s += order[i]->T;
        }
        if (out_reused_tokens) *out_reused_tokens = reused;
        if (slots.empty()) return CM_OK;
        cm_context *ctx = set->ctx;
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        return launch_slots(ctx, slots, set->L, set->H, set->d,
                            reinterpret_cast<cudaStream_t>(stream), withhold_warp, paged);
    });
}

}  // namespace

cm_status cm_render(const cm_set *set, void *k_out, void *v_out, int64_t capacity_tokens,
                    cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order) {
    return render_set(set, k_out, v_out, capacity_tokens, stream, out_seq_len, out_order, 0);
}

cm_status cm_render_many(const cm_render_job *jobs, int32_t n, cm_stream_t stream,
                         int64_t *out_seq_lens) {
    TraceRange trace("cm_render");
    return guarded([&]() -> cm_status {
        if (n < 0 || (n > 0 && !jobs)) return fail(CM_ERR_INVALID_ARG, "need n >= 0 jobs");
        cm_context *ctx = nullptr;
        bool has_shape = false;
        int32_t L = 0, H = 0, d = 0;
        std::vector<int64_t> totals((size_t)n);
        for (int32_t i = 0; i < n; ++i) {
            const cm_render_job &j = jobs[i];
            if (!j.set) return fail(CM_ERR_INVALID_ARG, "a job's set is NULL");
            if (j.capacity_tokens < 0) return fail(CM_ERR_INVALID_ARG, "capacity_tokens < 0");
            if (ctx && j.set->ctx != ctx)
                return fail(CM_ERR_INVALID_ARG, "sets belong to different contexts");
            ctx = j.set->ctx;
            int64_t total = 0;
            for (const auto &kv : j.set->items) total += kv.second->T;
            cm_status st = validate_outputs(j.k_out, j.v_out, j.capacity_tokens, total);
            if (st != CM_OK) return st;
            totals[(size_t)i] = total;
            if (total == 0) continue;
            if (!has_shape) {
                has_shape = true;
                L = j.set->L;
                H = j.set->H;
                d = j.set->d;
            } else if (j.set->L != L || j.set->H != H || j.set->d != d) {
                return fail(CM_ERR_SHAPE_MISMATCH, "sets of one cm_render_many call differ in shape");
            }
        }
        std::vector<Slot> slots;
        for (int32_t i = 0; i < n; ++i) {
            const cm_render_job &j = jobs[i];
            int64_t s = 0;
            for (const auto &r : canonical_order(j.set)) {
                slots.push_back({r->k, r->v, r->T, s, j.k_out, j.v_out, j.capacity_tokens});
                s += r->T;
            }
        }
        if (out_seq_lens)
            for (int32_t i = 0; i < n; ++i) out_seq_lens[i] = totals[(size_t)i];
        if (slots.empty()) return CM_OK;
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        return launch_slots(ctx, slots, L, H, d, reinterpret_cast<cudaStream_t>(stream));
    });
}

cm_status cm_set_contains(const cm_set *set, const cm_id *ids, int64_t n, uint8_t *out_present) {
    if (!set) return fail(CM_ERR_INVALID_ARG, "set is NULL");
    if (n < 0 || (n > 0 && (!ids || !out_present)))
        return fail(CM_ERR_INVALID_ARG, "need n >= 0 ids and an output array");
    for (int64_t i = 0; i < n; ++i)
        out_present[i] = set->items.count(key_of(ids[i])) ? 1 : 0;
    return CM_OK;
}

cm_status cm_set_leq(const cm_set *a, const cm_set *b, int32_t *out) {
    if (!a || !b || !out) return fail(CM_ERR_INVALID_ARG, "a, b or out is NULL");
    int32_t leq = 1;
    for (const auto &kv : a->items)
        if (!b->items.count(kv.first)) {
            leq = 0;
            break;
        }
    *out = leq;
    return CM_OK;
}

cm_status cm_render_incremental(const cm_set *set, void *k_out, void *v_out,
                                int64_t capacity_tokens, const cm_id *prev_order, int64_t prev_n,
                                cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order,
                                int64_t *out_reused_tokens) {
    return render_set(set, k_out, v_out, capacity_tokens, stream, out_seq_len, out_order, 0,
                      prev_order, prev_n, out_reused_tokens);
}

cm_status cm_render_paged(const cm_set *set, const cm_paged_cache *out, cm_stream_t stream,
                          int64_t *out_seq_len, cm_id *out_order) {
    if (!out) return fail(CM_ERR_INVALID_ARG, "paged cache descriptor is NULL");
    if (out->table_entries < 0 || out->block_size < 1)
        return fail(CM_ERR_INVALID_ARG, "table_entries < 0 or block_size < 1");
    if (out->table_entries > INT64_MAX / out->block_size)
        return fail(CM_ERR_INVALID_ARG, "table capacity overflows");
    return render_set(set, out->k_pool, out->v_pool, out->table_entries * out->block_size, stream,
                      out_seq_len, out_order, 0, nullptr, 0, nullptr, out);
}

cm_status cm_testing_render_withheld_load(const cm_set *set, void *k_out, void *v_out,
                                          int64_t capacity_tokens, cm_stream_t stream) {
    return render_set(set, k_out, v_out, capacity_tokens, stream, nullptr, nullptr, 1);
}

cm_status cm_testing_bounds_violations(int32_t device, uint64_t *out_count, int32_t *out_enabled) {
    return guarded([&]() -> cm_status {
        if (!out_count || !out_enabled) return fail(CM_ERR_INVALID_ARG, "out_count or out_enabled is NULL");
        DeviceScope scope(device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        CM_CUDA_TRY(cudaDeviceSynchronize(), "device synchronisation");
        unsigned int render = 0, hash = 0;
        CM_CUDA_TRY(cm::take_render_bounds_violations(&render), "render violation count");
        CM_CUDA_TRY(cm::take_hash_bounds_violations(&hash), "content-address violation count");
        *out_count = (uint64_t)render + hash;
#ifdef CM_DEBUG_BOUNDS
        *out_enabled = 1;
#else
        *out_enabled = 0;
#endif
        return CM_OK;
    });
}

cm_status cm_context_check(cm_context *ctx, cm_stream_t stream) {
    return guarded([&]() -> cm_status {
        if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        return take_device_error(ctx, reinterpret_cast<cudaStream_t>(stream));
    });
}

cm_status cm_bagmerge(cm_context *ctx, const cm_fragment *frags, int32_t n, void *k_out,
                      void *v_out, int64_t capacity_tokens, cm_stream_t stream,
                      int64_t *out_seq_len) {
    TraceRange trace("cm_bagmerge");
    return guarded([&]() -> cm_status {
        if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
        if (!frags || n < 1) return fail(CM_ERR_INVALID_ARG, "need n >= 1 fragments");
        if (capacity_tokens < 0) return fail(CM_ERR_INVALID_ARG, "capacity_tokens < 0");
        int64_t total = 0;
        for (int32_t i = 0; i < n; ++i) {
            cm_status st = validate_fragment(&frags[i]);
            if (st != CM_OK) return st;
            if (frags[i].num_layers != frags[0].num_layers ||
                frags[i].num_kv_heads != frags[0].num_kv_heads ||
                frags[i].head_dim != frags[0].head_dim)
                return fail(CM_ERR_SHAPE_MISMATCH, "fragments have different shapes");
            total += frags[i].seq_len;
        }
        cm_status st = validate_outputs(k_out, v_out, capacity_tokens, total);
        if (st != CM_OK) return st;
        std::vector<Slot> slots;
        int64_t s = 0;
        for (int32_t i = 0; i < n; ++i) {
            slots.push_back({frags[i].k, frags[i].v, frags[i].seq_len, s, k_out, v_out,
                             capacity_tokens});
            s += frags[i].seq_len;
        }
        if (out_seq_len) *out_seq_len = total;
        std::lock_guard<std::mutex> lock(ctx->mu);
        DeviceScope scope(ctx->device);
        if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
        return launch_slots(ctx, slots, frags[0].num_layers, frags[0].num_kv_heads,
                            frags[0].head_dim, reinterpret_cast<cudaStream_t>(stream));
    });
}

}  // extern "C"

// Helpers for the allocation-free content-address entry point (blake2s_tree.cu).
namespace cm {

TreeParams make_tree_params(int32_t L, int32_t H, int32_t d, int32_t T) {
    return tree_params(L, H, d, T);
}

cm_status check_fragment(const cm_fragment *f) { return validate_fragment(f); }

cm_status report_error(cm_status st, const char *msg) { return fail(st, msg); }

}  // namespace cm
