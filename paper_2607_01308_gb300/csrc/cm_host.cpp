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
    int leaf_blocks_per_sm = 0;   // leaf-hash blocks resident on one SM at once
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
    // cm_ingest_render: the stream its overlapped render runs on and the two events that
    // order it after the caller's stream and the caller's stream after it (made on first use)
    cudaStream_t side = nullptr;
    cudaEvent_t side_begin = nullptr, side_end = nullptr, side_keys = nullptr;
    int32_t overlap = 1;         // cm_context_set_overlap: 1 render beside the hash when possible
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

// Reads a small device result (`bytes` at `src`) into ctx->h_pinned + host_off, enqueued
// on `stream`: stored by the SMs through the buffer's mapped address when everything is
// 4-byte granular (so the read does not wait behind bulk device-to-host copies of other
// streams on the copy engine), else by a copy.
cudaError_t read_small_at(cm_context *ctx, size_t host_off, const void *src, size_t bytes,
                          cudaStream_t stream) {
    if (ctx->h_pinned_dev && bytes % 4 == 0 && host_off % 4 == 0 &&
        (reinterpret_cast<uintptr_t>(src) & 3u) == 0) {
        if (ctx->timing) ++ctx->aux_launches;
        return cm::launch_readback(static_cast<uint8_t *>(ctx->h_pinned_dev) + host_off, src, bytes,
                                   stream);
    }
    return cudaMemcpyAsync(ctx->h_pinned + host_off, src, bytes, cudaMemcpyDeviceToHost, stream);
}

cudaError_t read_small(cm_context *ctx, const void *src, size_t bytes, cudaStream_t stream) {
    return read_small_at(ctx, 0, src, bytes, stream);
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

// The scratch of one content-address pass over n fragments (Section 4.3; Algorithm 2,
// Id): device [roots n x 16][Q of fragment 0]...[Q of fragment n-1][arrival counters of
// the nodes at levels >= 2][the levels below each root]; the pinned host buffer receives
// [roots][Q ...] at the same offsets.
struct DigestPlan {
    struct Frag {
        std::vector<uint64_t> sizes;     // nodes per level, leaves first; the last is the root
        std::vector<size_t> level_off;   // device offsets of the levels below the root
        size_t q_off = 0, arr_off = 0;
        uint64_t plane = 0, stream_bytes = 0;
        int32_t rl = 0;
        cm::TreeParams tp;
    };
    std::vector<Frag> f;
    size_t roots_bytes = 0, host_bytes = 0, zero_end = 0, dev_bytes = 0;
};

cm_status plan_digest(cm_context *ctx, const cm_fragment *const *frags, size_t n, DigestPlan &plan) {
    plan.f.assign(n, DigestPlan::Frag());
    plan.roots_bytes = n * 16;
    size_t off = plan.roots_bytes;
    for (size_t i = 0; i < n; ++i) {
        const cm_fragment *f = frags[i];
        DigestPlan::Frag &l = plan.f[i];
        l.rl = routing_layer_for(ctx, f->num_layers);
        if (l.rl >= f->num_layers) return fail(CM_ERR_INVALID_ARG, "routing layer >= num_layers");
        l.plane = (uint64_t)f->num_kv_heads * f->seq_len * f->head_dim * 2;
        l.stream_bytes = 2ull * f->num_layers * l.plane;
        l.sizes.assign(1, ceil_div(l.stream_bytes, cm::kLeafBytes));
        while (l.sizes.size() == 1 || l.sizes.back() > 1)
            l.sizes.push_back(ceil_div(l.sizes.back(), cm::kFanout));
        if (l.sizes.size() > (size_t)cm::kMaxLevels)
            return fail(CM_ERR_UNSUPPORTED, "fragment too large for the hash tree depth");
        l.q_off = off;
        off += (size_t)f->seq_len * 8;
        l.tp = tree_params(f->num_layers, f->num_kv_heads, f->head_dim, f->seq_len);
    }
    plan.host_bytes = off;   // roots and norm keys
    // the arrival counters follow the norm keys, so that one memset zeroes both
    for (size_t i = 0; i < n; ++i) {
        plan.f[i].arr_off = off;
        for (size_t k = 2; k < plan.f[i].sizes.size(); ++k) off += (size_t)plan.f[i].sizes[k] * 4;
    }
    plan.zero_end = off;
    off = (off + 255) & ~(size_t)255;
    for (size_t i = 0; i < n; ++i) {
        DigestPlan::Frag &l = plan.f[i];
        for (size_t k = 0; k + 1 < l.sizes.size(); ++k) {   // the root goes to the roots area
            l.level_off.push_back(off);
            off += ((size_t)l.sizes[k] * cm::kDigestBytes + 255) & ~(size_t)255;
        }
    }
    plan.dev_bytes = off;
    return CM_OK;
}

// Enqueues a planned pass on `stream` (the scratch already holds plan.dev_bytes and
// plan.host_bytes): the leaf launches of up to kMaxLeafGroup fragments each (with the
// norm keys when with_norms), the tree levels above the leaves (level 1, then the levels
// above it: two launches per kMaxGroup fragments), and the results' way to the pinned
// buffer. When the buffer is mapped, the kernels that hash the roots store them there
// directly and only the norm keys are read back; otherwise roots and keys are copied.
cm_status enqueue_digest(cm_context *ctx, const DigestPlan &plan, const cm_fragment *const *frags,
                         size_t n, cudaStream_t stream, bool with_norms) {
    uint8_t *base = ctx->d_scratch;
    uint8_t *roots = ctx->h_pinned_dev ? static_cast<uint8_t *>(ctx->h_pinned_dev) : base;
    CM_CUDA_TRY(cudaMemsetAsync(base + plan.roots_bytes, 0, plan.zero_end - plan.roots_bytes, stream),
                "zeroing the norm keys and arrival counters");
    std::unique_ptr<cm::LeafGroup> grp(new cm::LeafGroup);
    for (size_t g0 = 0; g0 < n; g0 += (size_t)cm::kMaxLeafGroup) {
        const size_t gn = std::min(n - g0, (size_t)cm::kMaxLeafGroup);
        std::memset(grp.get(), 0, sizeof(cm::LeafGroup));
        grp->count = (uint32_t)gn;
        for (size_t q = 0; q < gn; ++q) {
            const cm_fragment *f = frags[g0 + q];
            const DigestPlan::Frag &l = plan.f[g0 + q];
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
        const cm::LeafPhases phases = with_norms ? cm::LeafPhases::kBoth : cm::LeafPhases::kLeaves;
        CM_CUDA_TRY(timed_launch(ctx, kTimeLeaf, stream,
                                 [&] { return cm::launch_leaf_hash_group(*grp, stream, phases); }),
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
        const DigestPlan::Frag &l = plan.f[i];
        const uint32_t c = top->count;
        cm::TreeTopFragment &tf = top->frag[c];
        tf.levels = (uint32_t)l.sizes.size();
        size_t a_off = l.arr_off;
        for (size_t k = 0; k < l.sizes.size(); ++k) {
            tf.size[k] = l.sizes[k];
            tf.level[k] = (k + 1 == l.sizes.size()) ? roots + 16 * i : base + l.level_off[k];
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
    if (!ctx->h_pinned_dev)
        CM_CUDA_TRY(read_small_at(ctx, 0, base, with_norms ? plan.host_bytes : plan.roots_bytes, stream),
                    "digest copy");
    else if (with_norms)
        CM_CUDA_TRY(read_small_at(ctx, plan.roots_bytes, base + plan.roots_bytes,
                                  plan.host_bytes - plan.roots_bytes, stream),
                    "norm-key copy");
    return CM_OK;
}

// After the stream reached the end of an enqueued pass: ids (and norm keys, if Qs).
void collect_digest(const cm_context *ctx, const DigestPlan &plan, const cm_fragment *const *frags,
                    size_t n, cm_id *ids, std::vector<uint64_t> *Qs) {
    for (size_t i = 0; i < n; ++i) {
        std::memcpy(ids[i].b, ctx->h_pinned + 16 * i, 16);
        if (Qs) {
            Qs[i].resize((size_t)frags[i]->seq_len);
            std::memcpy(Qs[i].data(), ctx->h_pinned + plan.f[i].q_off, (size_t)frags[i]->seq_len * 8);
        }
    }
}

// Id(C) and Q[t] of n fragments in one pass and one synchronisation of `stream`.
// Caller holds ctx->mu and the device scope.
cm_status fragments_digest(cm_context *ctx, const cm_fragment *const *frags, size_t n,
                           cudaStream_t stream, cm_id *ids, std::vector<uint64_t> *Qs) {
    DigestPlan plan;
    cm_status st = plan_digest(ctx, frags, n, plan);
    if (st == CM_OK) st = ensure_scratch(ctx, plan.dev_bytes, plan.host_bytes);
    if (st == CM_OK) st = enqueue_digest(ctx, plan, frags, n, stream, true);
    if (st != CM_OK) return st;
    CM_CUDA_TRY(cudaStreamSynchronize(stream), "ingest synchronisation");
    collect_digest(ctx, plan, frags, n, ids, Qs);
    return CM_OK;
}

// Enqueues Q[t] of n fragments alone (Eq. rho) on `stream`: one launch of the norm-key
// row threads per kMaxLeafGroup fragments (they read only K[l*]) into device scratch at
// dev_off (q_off[i] after it for fragment i; zeroed first), then a copy to the pinned
// buffer at host_off (same relative offsets).
cm_status enqueue_norm_keys(cm_context *ctx, const cm_fragment *const *frags, size_t n,
                            cudaStream_t stream, size_t dev_off, size_t host_off,
                            const std::vector<size_t> &q_off, size_t bytes) {
    uint8_t *base = ctx->d_scratch + dev_off;
    CM_CUDA_TRY(cudaMemsetAsync(base, 0, bytes, stream), "zeroing the norm keys");
    std::unique_ptr<cm::LeafGroup> grp(new cm::LeafGroup);
    for (size_t g0 = 0; g0 < n; g0 += (size_t)cm::kMaxLeafGroup) {
        const size_t gn = std::min(n - g0, (size_t)cm::kMaxLeafGroup);
        std::memset(grp.get(), 0, sizeof(cm::LeafGroup));
        grp->count = (uint32_t)gn;
        for (size_t q = 0; q < gn; ++q) {
            const cm_fragment *f = frags[g0 + q];
            cm::LeafLaunch &a = grp->frag[q];
            a.k = static_cast<const uint8_t *>(f->k);
            a.v = static_cast<const uint8_t *>(f->v);
            a.plane_bytes = (uint64_t)f->num_kv_heads * f->seq_len * f->head_dim * 2;
            a.stream_bytes = 2ull * f->num_layers * a.plane_bytes;
            a.num_leaves = ceil_div(a.stream_bytes, cm::kLeafBytes);
            a.norm_begin = 2ull * (uint64_t)routing_layer_for(ctx, f->num_layers) * a.plane_bytes;
            a.row_bytes = (uint32_t)f->head_dim * 2;
            a.seq_len = (uint32_t)f->seq_len;
            a.norm_key = reinterpret_cast<unsigned long long *>(base + q_off[g0 + q]);
            a.tree = tree_params(f->num_layers, f->num_kv_heads, f->head_dim, f->seq_len);
            grp->block_begin[q + 1] =
                grp->block_begin[q] + ceil_div(a.num_leaves, (uint64_t)cm::kLeafBlockThreads);
        }
        if (grp->block_begin[gn] > 0x7FFFFFFFull)
            return fail(CM_ERR_UNSUPPORTED, "leaf-hash launch exceeds 2^31 - 1 blocks");
        CM_CUDA_TRY(cm::launch_leaf_hash_group(*grp, stream, cm::LeafPhases::kNormKeys),
                    "norm-key launch");
        if (ctx->timing) ++ctx->aux_launches;
    }
    CM_CUDA_TRY(read_small_at(ctx, host_off, base, bytes, stream), "norm-key copy");
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
                       const cm_paged_cache *paged = nullptr, const cm::RenderWidth *width = nullptr) {
    // no width: the context's. The failure-injection hook withholds a TMA copy, so it runs
    // the half-SM kernel (the TMA kernels are the ones that wait).
    const cm::RenderWidth warps =
        withhold_warp ? cm::RenderWidth::kHalf
                      : width ? *width
                              : (ctx->render_warps == 8 ? cm::RenderWidth::kHalf : cm::RenderWidth::kFull);
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

// S = sum of Q[t] over the last t_star of a fragment's T positions (the integer form of
// rho, Eq. rho, up to the common factor 2^-20 / (H T*)).
unsigned __int128 tail_sum(const std::vector<uint64_t> &Q, int64_t T, int32_t H, int64_t t_star) {
    // each Q[t] is at most H (2^44 - 1): when H T* (2^44 - 1) < 2^64 the tail sum cannot
    // wrap in 64 bits, and a plain 64-bit sum (which vectorises) is exact
    const uint64_t *q = Q.data() + (T - t_star);
    if ((unsigned __int128)H * (uint64_t)t_star * ((1ull << 44) - 1) < ((unsigned __int128)1 << 64)) {
        uint64_t s64 = 0;
        for (int64_t t = 0; t < t_star; ++t) s64 += q[t];
        return s64;
    }
    unsigned __int128 S = 0;
    for (int64_t t = 0; t < t_star; ++t) S += q[t];
    return S;
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
    for (auto &r : recs) keyed.push_back({tail_sum(r->Q, r->T, r->H, t_star), key_of(r->id), r});
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

// Validation of n deliveries, delivery i into sets[i]: all sets from one context (*ctx),
// each delivery of its set's shape (an empty set takes its first delivery's), a valid
// routing layer. fp receives the descriptors.
cm_status validate_deliveries(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                              cm_context **ctx_out, std::vector<const cm_fragment *> &fp) {
    cm_context *ctx = sets[0]->ctx;
    struct Shape {
        bool has;
        int32_t L, H, d;
    };
    std::unordered_map<const cm_set *, Shape> shape;
    fp.assign((size_t)n, nullptr);
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
    *ctx_out = ctx;
    return CM_OK;
}

// Where delivery i's id and norm key come from: a stored record it is byte-identical to
// (rec[i]), an earlier delivery of the call (from[i] >= 0), or the content-address pass
// (hashed_as[i] indexes hashed_ids / hashed_Q).
struct DeliverySources {
    std::vector<std::shared_ptr<const Record>> rec;
    std::vector<int32_t> from;
    std::vector<size_t> hashed_as;
    std::vector<const cm_fragment *> to_hash;
};

DeliverySources hash_everything(size_t n, const std::vector<const cm_fragment *> &fp) {
    DeliverySources src;
    src.rec.assign(n, nullptr);
    src.from.assign(n, -1);
    src.hashed_as.resize(n);
    for (size_t i = 0; i < n; ++i) {
        src.hashed_as[i] = i;
        src.to_hash.push_back(fp[i]);
    }
    return src;
}

// The insertions of Ingest (Algorithm 2) in delivery order, once every delivery's id and
// norm key are known: a delivery whose id its set already holds (before the call or from
// an earlier delivery of it) is absorbed; with verify_bytes_on_hit its bytes are compared
// with the stored record's first (CM_ERR_COLLISION if they differ: the deliveries before
// it stay inserted). hashed_Q is consumed.
cm_status insert_deliveries(cm_context *ctx, cm_set *const *sets,
                            const std::vector<const cm_fragment *> &fp, cudaStream_t cs,
                            const DeliverySources &src, const std::vector<cm_id> &hashed_ids,
                            std::vector<std::vector<uint64_t>> &hashed_Q, cm_id *out_ids,
                            int32_t *out_absorbed) {
    const size_t n = fp.size();
    // ids in delivery order; Qsrc[i] is where delivery i's norm key lives once delivery i
    // has been processed (its own record, a record it matched, or a hashed result)
    std::vector<cm_id> ids(n);
    std::vector<const std::vector<uint64_t> *> Qsrc(n, nullptr);
    for (size_t i = 0; i < n; ++i) {
        cm_set *set = sets[i];
        const cm_fragment *f = fp[i];
        std::vector<uint64_t> *own = nullptr;
        if (src.rec[i]) {
            ids[i] = src.rec[i]->id;
            Qsrc[i] = &src.rec[i]->Q;
        } else if (src.from[i] >= 0) {
            ids[i] = ids[(size_t)src.from[i]];
            Qsrc[i] = Qsrc[(size_t)src.from[i]];
        } else {
            ids[i] = hashed_ids[src.hashed_as[i]];
            own = &hashed_Q[src.hashed_as[i]];
            Qsrc[i] = own;
        }
        if (out_ids) out_ids[i] = ids[i];
        const IdKey key = key_of(ids[i]);
        auto it = set->items.find(key);
        if (it != set->items.end()) {
            // a byte match against this very record needs no second look at the bytes
            if (ctx->verify && src.rec[i] != it->second) {
                bool equal = false;
                cm_status st = bytes_equal(ctx, f, *it->second, cs, &equal);
                if (st != CM_OK) return st;
                if (!equal) return fail(CM_ERR_COLLISION, "content address hit with different bytes");
            }
            if (out_absorbed) out_absorbed[i] = 1;
            continue;
        }
        auto rec = std::make_shared<Record>();
        rec->id = ids[i];
        rec->L = f->num_layers;
        rec->H = f->num_kv_heads;
        rec->T = f->seq_len;
        rec->d = f->head_dim;
        rec->k = f->k;
        rec->v = f->v;
        if (own)
            rec->Q = std::move(*own);
        else
            rec->Q = *Qsrc[i];
        Qsrc[i] = &rec->Q;
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

// Ingest (Algorithm 2) of the validated deliveries fp, delivery i into sets[i]: one GPU
// pass for all of them (after the re-delivery fast path, when it is on), then the
// insertions in delivery order. Caller holds ctx->mu and the device scope.
cm_status ingest_validated(cm_context *ctx, cm_set *const *sets,
                           const std::vector<const cm_fragment *> &fp, cudaStream_t cs,
                           cm_id *out_ids, int32_t *out_absorbed) {
    const size_t n = fp.size();
    DeliverySources src;
    if (ctx->dedup_bytes) {
        // deliveries byte-identical to a known fragment take its id and norm key and are
        // not hashed
        cm_status st = find_redeliveries(ctx, sets, fp, cs, src.rec, src.from);
        if (st != CM_OK) return st;
        src.hashed_as.assign(n, 0);
        for (size_t i = 0; i < n; ++i)
            if (!src.rec[i] && src.from[i] < 0) {
                src.hashed_as[i] = src.to_hash.size();
                src.to_hash.push_back(fp[i]);
            }
    } else {
        src = hash_everything(n, fp);
    }
    std::vector<cm_id> hashed_ids(src.to_hash.size());
    std::vector<std::vector<uint64_t>> hashed_Q(src.to_hash.size());
    if (!src.to_hash.empty()) {
        cm_status st = fragments_digest(ctx, src.to_hash.data(), src.to_hash.size(), cs,
                                        hashed_ids.data(), hashed_Q.data());
        if (st != CM_OK) return st;
    }
    return insert_deliveries(ctx, sets, fp, cs, src, hashed_ids, hashed_Q, out_ids, out_absorbed);
}

// Ingest (Algorithm 2) of n deliveries, delivery i into sets[i] (several entries
// may name one set). Nothing is inserted if validation fails.
cm_status ingest_deliveries(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                            cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed) {
    if (n == 0) return CM_OK;
    cm_context *ctx = nullptr;
    std::vector<const cm_fragment *> fp;
    cm_status st = validate_deliveries(sets, frags, n, &ctx, fp);
    if (st != CM_OK) return st;
    std::lock_guard<std::mutex> lock(ctx->mu);
    DeviceScope scope(ctx->device);
    if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
    return ingest_validated(ctx, sets, fp, reinterpret_cast<cudaStream_t>(stream), out_ids,
                            out_absorbed);
}

// dst := dst u src (Eq. setunion); shapes already checked. On equal ids dst keeps its
// record (the bytes are equal).
void union_into(cm_set *dst, const cm_set *src) {
    for (const auto &kv : src->items) dst->items.emplace(kv.first, kv.second);
    if (!dst->has_shape && src->has_shape) {
        dst->has_shape = true;
        dst->L = src->L;
        dst->H = src->H;
        dst->d = src->d;
    }
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
        ctx->leaf_blocks_per_sm = cm::leaf_hash_blocks_per_sm();
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
        if (ctx->side) cudaStreamDestroy(ctx->side);
        if (ctx->side_begin) cudaEventDestroy(ctx->side_begin);
        if (ctx->side_end) cudaEventDestroy(ctx->side_end);
        if (ctx->side_keys) cudaEventDestroy(ctx->side_keys);
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

cm_status cm_context_set_overlap(cm_context *ctx, int32_t mode) {
    if (!ctx) return fail(CM_ERR_INVALID_ARG, "context is NULL");
    if (mode != 0 && mode != 1) return fail(CM_ERR_INVALID_ARG, "overlap mode must be 0 or 1");
    std::lock_guard<std::mutex> lock(ctx->mu);
    ctx->overlap = mode;
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
        union_into(dst, src);
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

// Slots of the set's canonical order at offsets s = exclusive prefix sums of T, into
// one contiguous output; *order receives the records in that order.
std::vector<Slot> canonical_slots(const cm_set *set, void *k_out, void *v_out, int64_t capacity,
                                  std::vector<std::shared_ptr<const Record>> *order) {
    *order = canonical_order(set);
    std::vector<Slot> slots;
    int64_t s = 0;
    for (const auto &r : *order) {
        slots.push_back({r->k, r->v, r->T, s, k_out, v_out, capacity});
        s += r->T;
    }
    return slots;
}

// A render beside the leaf hash (cm_ingest_render) whose fragments hold at least this
// many bytes takes the 4-warp TMA kernel, a smaller one the register kernel with one CTA
// per SM: measured on the Qwen3 shapes, the register kernel was the faster neighbour of
// the hash for 0.3 GB of fragments, the TMA kernel from 1.2 GB on.
constexpr uint64_t kBesideLargeBytes = 512ull << 20;

cm_status ensure_side_stream(cm_context *ctx) {
    if (!ctx->side) {
        // the highest priority: the render's CTAs, launched while the leaf hash's grid is
        // already queued, are dispatched as soon as any of its blocks retire
        int least = 0, greatest = 0;
        CM_CUDA_TRY(cudaDeviceGetStreamPriorityRange(&least, &greatest), "stream priorities");
        CM_CUDA_TRY(cudaStreamCreateWithPriority(&ctx->side, cudaStreamNonBlocking, greatest),
                    "side stream");
    }
    if (!ctx->side_begin)
        CM_CUDA_TRY(cudaEventCreateWithFlags(&ctx->side_begin, cudaEventDisableTiming), "side event");
    if (!ctx->side_end)
        CM_CUDA_TRY(cudaEventCreateWithFlags(&ctx->side_end, cudaEventDisableTiming), "side event");
    if (!ctx->side_keys)
        CM_CUDA_TRY(cudaEventCreateWithFlags(&ctx->side_keys, cudaEventDisableTiming), "side event");
    return CM_OK;
}

// cm_ingest_render (see include/cm.h). The norm keys of the deliveries are computed on
// the context's side stream while the content address runs on `stream`. Equal bytes give
// equal norm keys, so members of the prospective set whose integer tail sums S (Eq. rho),
// lengths and norm keys agree are taken for one fragment, and when the remaining S are
// pairwise distinct the canonical order of Algorithm 1 is decided before any id is known:
// the render then starts on the side stream (narrow CTAs) beside the rest of the content
// address. Once the ids are known the insertions and unions are made as usual; if the set
// that results does not hold exactly the fragments the render assumed, in that order
// (different fragments taken for one, or an address collision, which the paper excludes),
// it is rendered again after the first render.
cm_status ingest_render_impl(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                             cm_set *target, void *k_out, void *v_out, int64_t capacity,
                             cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed,
                             int64_t *out_seq_len, cm_id *out_order, int32_t *out_overlapped) {
    if (!target) return fail(CM_ERR_INVALID_ARG, "target set is NULL");
    if (capacity < 0) return fail(CM_ERR_INVALID_ARG, "capacity_tokens < 0");
    if (n < 0 || (n > 0 && (!frags || !sets)))
        return fail(CM_ERR_INVALID_ARG, "need n >= 0 fragments and their sets");
    for (int32_t i = 0; i < n; ++i)
        if (!sets[i]) return fail(CM_ERR_INVALID_ARG, "a set is NULL");
    if (out_overlapped) *out_overlapped = 0;
    cm_context *ctx = target->ctx;
    std::vector<const cm_fragment *> fp;
    if (n > 0) {
        cm_context *dctx = nullptr;
        cm_status st = validate_deliveries(sets, frags, n, &dctx, fp);
        if (st != CM_OK) return st;
        if (dctx != ctx) return fail(CM_ERR_INVALID_ARG, "sets belong to different contexts");
    }
    // the union sources: the sets the deliveries go to, other than the target, in order
    std::vector<cm_set *> sources;
    for (int32_t i = 0; i < n; ++i)
        if (sets[i] != target && std::find(sources.begin(), sources.end(), sets[i]) == sources.end())
            sources.push_back(sets[i]);
    bool has = false;
    int32_t L = 0, H = 0, d = 0;
    auto same_shape = [&](bool h, int32_t l, int32_t hh, int32_t dd) {
        if (!h) return true;
        if (!has) {
            has = true;
            L = l;
            H = hh;
            d = dd;
            return true;
        }
        return l == L && hh == H && dd == d;
    };
    bool one_shape = same_shape(target->has_shape, target->L, target->H, target->d);
    for (const cm_set *src : sources) one_shape = same_shape(src->has_shape, src->L, src->H, src->d) && one_shape;
    for (const cm_fragment *f : fp)
        one_shape = same_shape(true, f->num_layers, f->num_kv_heads, f->head_dim) && one_shape;
    if (!one_shape)
        return fail(CM_ERR_SHAPE_MISMATCH, "the target, the other sets and the deliveries of one "
                                           "cm_ingest_render call must share one shape");
    std::lock_guard<std::mutex> lock(ctx->mu);
    DeviceScope scope(ctx->device);
    if (!scope.ok()) return fail(CM_ERR_CUDA, "cannot select the CUDA device");
    const cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);

    // the one-after-the-other path: the re-delivery fast path compares bytes before any
    // hashing, and overlap mode 0 asks for it
    if (n == 0 || ctx->dedup_bytes || ctx->overlap == 0) {
        cm_status st = n > 0 ? ingest_validated(ctx, sets, fp, cs, out_ids, out_absorbed) : CM_OK;
        if (st != CM_OK) return st;
        for (const cm_set *src : sources) union_into(target, src);
        std::vector<std::shared_ptr<const Record>> order;
        const std::vector<Slot> slots = canonical_slots(target, k_out, v_out, capacity, &order);
        int64_t total = 0;
        for (const auto &r : order) total += r->T;
        st = validate_outputs(k_out, v_out, capacity, total);
        if (st != CM_OK) return st;
        if (out_seq_len) *out_seq_len = total;
        if (out_order)
            for (size_t i = 0; i < order.size(); ++i) out_order[i] = order[i]->id;
        if (slots.empty()) return CM_OK;
        return launch_slots(ctx, slots, target->L, target->H, target->d, cs);
    }

    // scratch: the content-address pass, then the norm keys (device and pinned host)
    DigestPlan plan;
    cm_status st = plan_digest(ctx, fp.data(), fp.size(), plan);
    if (st != CM_OK) return st;
    const size_t q_dev = (plan.dev_bytes + 255) & ~(size_t)255;
    const size_t q_host = (plan.host_bytes + 255) & ~(size_t)255;
    std::vector<size_t> q_off((size_t)n);
    size_t q_bytes = 0;
    for (int32_t i = 0; i < n; ++i) {
        q_off[(size_t)i] = q_bytes;
        q_bytes += (size_t)fp[(size_t)i]->seq_len * 8;
    }
    st = ensure_scratch(ctx, q_dev + q_bytes, q_host + q_bytes);
    if (st == CM_OK) st = ensure_side_stream(ctx);
    if (st != CM_OK) return st;
    CM_CUDA_TRY(cudaEventRecord(ctx->side_begin, cs), "side stream ordering");
    CM_CUDA_TRY(cudaStreamWaitEvent(ctx->side, ctx->side_begin, 0), "side stream ordering");
    // from here on, every way out (a C++ exception included) orders the caller's stream
    // after the side stream's work: explicitly through join(), else in the destructor
    struct SideJoin {
        cm_context *ctx;
        cudaStream_t cs;
        bool done = false;
        cudaError_t run() {
            done = true;
            cudaError_t e = cudaEventRecord(ctx->side_end, ctx->side);
            if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ctx->side_end, 0);
            return e;
        }
        ~SideJoin() {
            if (!done) run();
        }
    } side_join{ctx, cs};
    auto join = [&](cm_status prior) -> cm_status {
        const cudaError_t e = side_join.run();
        if (e != cudaSuccess && prior == CM_OK) return cuda_fail(e, "side stream ordering");
        return prior;
    };
    // The norm keys decide when the render can start. A leaf grid that leaves a block's room
    // on every SM (one partial wave) is launched first: the hash starts a few launches
    // earlier and the norm-key blocks still start at once beside it. A larger grid would
    // take every SM and hold back norm keys launched after it until its first wave retires.
    uint64_t leaf_blocks = 0;
    for (const DigestPlan::Frag &l : plan.f) leaf_blocks += ceil_div(l.sizes[0], (uint64_t)cm::kLeafBlockThreads);
    const bool digest_first =
        ctx->leaf_blocks_per_sm > 1 &&
        leaf_blocks <= (uint64_t)(ctx->leaf_blocks_per_sm - 1) * (uint64_t)ctx->num_sms;
    if (digest_first) {
        st = enqueue_digest(ctx, plan, fp.data(), fp.size(), cs, false);
        if (st != CM_OK) return join(st);
    }
    st = enqueue_norm_keys(ctx, fp.data(), fp.size(), ctx->side, q_dev, q_host, q_off, q_bytes);
    if (st != CM_OK) return join(st);
    cudaError_t e = cudaEventRecord(ctx->side_keys, ctx->side);
    if (e != cudaSuccess) return join(cuda_fail(e, "side stream ordering"));
    if (!digest_first) {
        st = enqueue_digest(ctx, plan, fp.data(), fp.size(), cs, false);
        if (st != CM_OK) return join(st);
    }
    e = cudaEventSynchronize(ctx->side_keys);
    if (e != cudaSuccess) return join(cuda_fail(e, "norm-key synchronisation"));
    std::vector<std::vector<uint64_t>> Qd((size_t)n);
    for (int32_t i = 0; i < n; ++i) {
        Qd[(size_t)i].resize((size_t)fp[(size_t)i]->seq_len);
        std::memcpy(Qd[(size_t)i].data(), ctx->h_pinned + q_host + q_off[(size_t)i],
                    (size_t)fp[(size_t)i]->seq_len * 8);
    }

    // the prospective set: the records of the target and of the sources (one per id),
    // then every delivery; distinct tail sums decide its order. Members with equal sums,
    // lengths and norm keys are taken for one fragment (byte-identical fragments always
    // agree so; a duplicate delivery is absorbed): the render uses the first of them, whose
    // bytes then equal those of whichever copy the set keeps. Equal sums with different
    // lengths or norm keys are a tie only the ids can break.
    bool spec = true;
    std::vector<Slot> spec_slots;
    struct Member {
        const void *k, *v;
        int64_t T;
        unsigned __int128 S;
        const std::vector<uint64_t> *Q;
        bool has_id;       // a record: its id; a delivery: known once hashed
        IdKey id;
        size_t delivery;
    };
    std::vector<Member> spec_members;
    {
        std::map<IdKey, std::shared_ptr<const Record>> have(target->items.begin(), target->items.end());
        for (const cm_set *src : sources) have.insert(src->items.begin(), src->items.end());
        int64_t t_star = INT64_MAX;
        for (const auto &kv : have) t_star = std::min<int64_t>(t_star, kv.second->T);
        for (const cm_fragment *f : fp) t_star = std::min<int64_t>(t_star, f->seq_len);
        std::vector<Member> m;
        for (const auto &kv : have) {
            const Record &r = *kv.second;
            m.push_back({r.k, r.v, r.T, tail_sum(r.Q, r.T, r.H, t_star), &r.Q, true, kv.first, 0});
        }
        for (size_t i = 0; i < fp.size(); ++i)
            m.push_back({fp[i]->k, fp[i]->v, fp[i]->seq_len,
                         tail_sum(Qd[i], fp[i]->seq_len, fp[i]->num_kv_heads, t_star), &Qd[i], false,
                         IdKey{}, i});
        // records first, then deliveries in order, within equal sums
        std::stable_sort(m.begin(), m.end(), [](const Member &a, const Member &b) { return a.S > b.S; });
        int64_t total = 0;
        for (const Member &x : m) {
            if (!spec_members.empty() && spec_members.back().S == x.S) {
                const Member &y = spec_members.back();
                if (y.T == x.T && *y.Q == *x.Q) continue;   // taken for the same fragment
                spec = false;
            }
            spec_members.push_back(x);
            total += x.T;
        }
        // an output the render would refuse: no speculation (the call then fails as
        // cm_render does, after the ingest); a small merge: the render follows the hash
        if (capacity < total || !k_out || !v_out || !aligned16(k_out) || !aligned16(v_out))
            spec = false;
        if (spec) {
            int64_t s = 0;
            for (const Member &x : spec_members) {
                spec_slots.push_back({x.k, x.v, x.T, s, k_out, v_out, capacity});
                s += x.T;
            }
            // beside the leaf hash: a narrow render, its kernel chosen by size
            const uint64_t frag_bytes = 2ull * (uint64_t)total * (uint64_t)L * (uint64_t)H * (uint64_t)d * 2;
            const cm::RenderWidth beside = frag_bytes >= kBesideLargeBytes
                                               ? cm::RenderWidth::kBeside
                                               : cm::RenderWidth::kBesideSmall;
            st = launch_slots(ctx, spec_slots, L, H, d, ctx->side, 0, nullptr, &beside);
            if (st != CM_OK) return join(st);
        }
    }
    e = cudaStreamSynchronize(cs);
    if (e != cudaSuccess) return join(cuda_fail(e, "ingest synchronisation"));
    std::vector<cm_id> ids((size_t)n);
    collect_digest(ctx, plan, fp.data(), fp.size(), ids.data(), nullptr);
    st = insert_deliveries(ctx, sets, fp, cs, hash_everything(fp.size(), fp), ids, Qd, out_ids,
                           out_absorbed);
    if (st != CM_OK) return join(st);
    for (const cm_set *src : sources) union_into(target, src);
    std::vector<std::shared_ptr<const Record>> order;
    const std::vector<Slot> slots = canonical_slots(target, k_out, v_out, capacity, &order);
    int64_t total = 0;
    for (const auto &r : order) total += r->T;
    st = validate_outputs(k_out, v_out, capacity, total);
    if (st != CM_OK) return join(st);
    if (out_seq_len) *out_seq_len = total;
    if (out_order)
        for (size_t i = 0; i < order.size(); ++i) out_order[i] = order[i]->id;
    // the render stands if the set holds exactly the members assumed, in the same order:
    // the same ids (so the same bytes, rendered from whichever copy) and lengths
    bool kept = spec && order.size() == spec_members.size();
    for (size_t i = 0; kept && i < order.size(); ++i) {
        const Member &x = spec_members[i];
        kept = key_of(order[i]->id) == (x.has_id ? x.id : key_of(ids[x.delivery])) && order[i]->T == x.T;
    }
    // no speculation, or not the set that resulted: render now, after anything before
    if (!kept && !slots.empty()) st = launch_slots(ctx, slots, target->L, target->H, target->d, ctx->side);
    st = join(st);
    if (st == CM_OK && out_overlapped) *out_overlapped = kept ? 1 : 0;
    return st;
}

}  // namespace

cm_status cm_render(const cm_set *set, void *k_out, void *v_out, int64_t capacity_tokens,
                    cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order) {
    return render_set(set, k_out, v_out, capacity_tokens, stream, out_seq_len, out_order, 0);
}

cm_status cm_ingest_render(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                           cm_set *target, void *k_out, void *v_out, int64_t capacity_tokens,
                           cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed,
                           int64_t *out_seq_len, cm_id *out_order, int32_t *out_overlapped) {
    TraceRange trace("cm_ingest_render");
    return guarded([&]() -> cm_status {
        return ingest_render_impl(sets, frags, n, target, k_out, v_out, capacity_tokens, stream,
                                  out_ids, out_absorbed, out_seq_len, out_order, out_overlapped);
    });
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
