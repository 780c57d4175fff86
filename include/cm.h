/*
 * cm.h - C ABI of the GB300 CanonicalMerge / LatentFragmentSet library (libcm.so).
 *
 * The library implements the data-parallel hot path of "Cache Merging as a
 * Convergent Replicated State for Multi-Agent Latent Reasoning":
 *
 *   Id(C)        content address of a KV-cache fragment          (Section 4.3; Algorithm 2, Id)
 *   Ingest(S,C)  S u {(Id(C), C)}, duplicates absorbed            (Algorithm 2, Ingest)
 *   Merge(S1,S2) set union                                        (Eq. setunion; Algorithm 2, Merge)
 *   Render(S)    CanonicalMerge of the set's fragments            (Algorithm 1; Algorithm 2, Render)
 *
 * Data layout. A fragment is one agent's legacy KV cache with the batch
 * dimension (always 1) dropped: K and V are two DEVICE buffers, each
 * [num_layers][num_kv_heads][seq_len][head_dim] bf16, contiguous, row-major,
 * K stored post-RoPE (the key at position t already rotated by R(t)).
 * A rendered cache is two caller-owned DEVICE buffers
 * [num_layers][num_kv_heads][capacity_tokens][head_dim] bf16 (row stride =
 * capacity_tokens); positions >= the rendered length are left untouched.
 *
 * Conventions fixed by this library where the paper leaves a choice:
 *   - content address: BLAKE2s tree hash (RFC 7693; 1024-byte leaves, fanout 16,
 *     16-byte digests, shapes and dtype in the salt, seq_len in the personalisation)
 *     of the byte stream K[0],V[0],...,K[L-1],V[L-1];
 *   - routing layer l* 0-indexed, default floor(L/2); the K-norm score is carried
 *     as an exact integer key (per-row fp64 norm, quantised to 2^-20);
 *   - canonical order: descending score, ties by descending id read big-endian;
 *   - RoPE re-encoding uses the rotate-half pairing (j, j + head_dim/2),
 *     frequency theta^(-2j/head_dim); the slot at offset 0 is a byte copy; V is a
 *     byte copy. Re-rotated K is the fp64 rotation rounded once to bf16, bit for bit.
 *
 * Errors. Every call validates all arguments before it enqueues any GPU work and
 * returns a cm_status; no C++ exception crosses this boundary and nothing aborts.
 * cm_last_error_message() gives a thread-local description of the last failure.
 *
 * Threading. Calls on one context are serialised by a lock inside the context.
 * A set must not be modified (ingest, union, destroy) while another thread uses it.
 */
#ifndef CM_H_
#define CM_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define CM_ABI_VERSION 5

/* Same type as cudaStream_t (a CUDA runtime stream handle); NULL is the legacy default stream. */
typedef struct CUstream_st *cm_stream_t;

typedef enum cm_status {
    CM_OK = 0,
    CM_ERR_INVALID_ARG = 1,     /* null pointer, non-positive size, unsupported head_dim, bad routing layer */
    CM_ERR_SHAPE_MISMATCH = 2,  /* (layers, kv_heads, head_dim) differ from the set's */
    CM_ERR_CAPACITY = 3,        /* rendered length exceeds capacity_tokens */
    CM_ERR_ALIGNMENT = 4,       /* a device buffer is not 16-byte aligned */
    CM_ERR_COLLISION = 5,       /* verify_bytes_on_hit: equal id, different bytes */
    CM_ERR_CUDA = 6,            /* a CUDA runtime call failed (message has the CUDA error text) */
    CM_ERR_OOM = 7,             /* host or device allocation failed */
    CM_ERR_TIMEOUT = 8,         /* a bounded device-side wait ran out (reported by cm_context_check) */
    CM_ERR_UNSUPPORTED = 9      /* too many fragments for one render launch group, or shape beyond limits */
} cm_status;

/* 16-byte content address: the BLAKE2s tree root digest, in digest byte order. */
typedef struct cm_id {
    uint8_t b[16];
} cm_id;

/* One KV-cache fragment. k and v are DEVICE pointers, 16-byte aligned, each
 * [num_layers][num_kv_heads][seq_len][head_dim] bf16 contiguous. Limits:
 * 1 <= num_layers, num_kv_heads <= 65535; seq_len >= 1; head_dim a power of two
 * in [16, 512]. The library only reads them. */
typedef struct cm_fragment {
    int32_t num_layers;
    int32_t num_kv_heads;
    int32_t seq_len;
    int32_t head_dim;
    const void *k;
    const void *v;
} cm_fragment;

typedef struct cm_context cm_context;
typedef struct cm_set cm_set;

/* Library and ABI version (CM_ABI_VERSION). */
int32_t cm_abi_version(void);

/* Create a context on CUDA device `device`.
 *   rope_theta          RoPE base theta (> 0), e.g. 1e6 for Qwen3 (Section 4.1)
 *   routing_layer       l* (0-indexed); < 0 selects floor(num_layers / 2) per fragment (Section 4.3)
 *   verify_bytes_on_hit nonzero: when an ingested fragment's id is already in the set,
 *                       compare its bytes with the stored fragment on the device and
 *                       return CM_ERR_COLLISION if they differ (the paper assumes a
 *                       collision-resistant hash, Section 4.3, so this never fires)
 * The context owns device scratch for hashing, grown on demand and freed by
 * cm_context_destroy. *out receives the handle. */
cm_status cm_context_create(int32_t device, double rope_theta, int32_t routing_layer,
                            int32_t verify_bytes_on_hit, cm_context **out);

/* Destroy a context. All sets created from it must have been destroyed. NULL is a no-op. */
cm_status cm_context_destroy(cm_context *ctx);

/* Create an empty LatentFragmentSet bound to ctx (Section 4.4). */
cm_status cm_set_create(cm_context *ctx, cm_set **out);

/* Destroy a set (NULL is a no-op). Fragment buffers are borrowed, never freed here. */
cm_status cm_set_destroy(cm_set *set);

/* Id(C) of Algorithm 2 and the routing-layer norm key of Eq. rho, without a set.
 * Runs the hash kernels on `stream` and returns after the result reached the host
 * (the stream is synchronised).
 *   out_id        receives the 16-byte content address (required)
 *   out_norm_key  nullable HOST array of frag->seq_len uint64: Q[t] = sum over kv heads of
 *                 round-half-even(2^20 * ||K[l*][h][t][:]||_2), each term saturated at 2^44-1 */
cm_status cm_fragment_id(cm_context *ctx, const cm_fragment *frag, cm_stream_t stream,
                         cm_id *out_id, uint64_t *out_norm_key);

/* Allocation-free variant of cm_fragment_id (the paper has no counterpart; this is
 * for callers that cannot allocate device memory: a serving engine that has
 * handed nearly all of the GPU's memory to its own paged KV-cache pool, where a
 * surprise cudaMalloc would fail or fragment that pool, or code that routes every
 * device allocation through its own allocator and forbids the CUDA one).
 * It computes the same id and norm key as cm_fragment_id on the calling thread's
 * current device, asynchronously on `stream`, and calls no cudaMalloc, cudaFree or
 * other allocating routine: the tree levels below the root live in a static device
 * array of 17.25 MiB that every GPU that loads libcm.so holds until the process
 * exits.
 *   routing_layer  l* (0-indexed); < 0 selects floor(num_layers / 2)
 *   id_out         DEVICE, 16-byte aligned, 16 bytes: receives the id
 *   norm_key_out   DEVICE, 8-byte aligned, seq_len uint64: receives Q[t] (it is zeroed
 *                  on `stream` first, then accumulated)
 * Limit: the fragment's K and V bytes (2 * L * H * T * d * 2) must not exceed 1 GiB;
 * larger fragments return CM_ERR_UNSUPPORTED (use cm_fragment_id).
 * Every call looks the array's device address up (cudaGetSymbolAddress, on the calling
 * thread's current device) and keeps no copy of it, so a device reset or another context
 * on the device never leaves a stale address in use.
 * Every call shares the one array: calls whose GPU work overlaps (on different
 * streams, or from several threads) race and corrupt each other's results; order
 * them on one stream or synchronise between them. Returns after enqueueing. */
cm_status cm_fragment_id_static(const cm_fragment *frag, int32_t routing_layer,
                                cm_stream_t stream, void *id_out, uint64_t *norm_key_out);

/* Ingest(S, C) of Algorithm 2: content-address the fragment (one pass over its
 * bytes on `stream`, which is synchronised before return, because membership is
 * decided on the host) and insert it keyed by its id. A fragment whose id is
 * already present is absorbed (*out_absorbed = 1) and the set is unchanged.
 * The set BORROWS frag->k and frag->v: they must stay allocated and unmodified
 * while the set (or any set it was unioned into) holds the id. The first
 * fragment fixes the set's (num_layers, num_kv_heads, head_dim); later ones must
 * match (CM_ERR_SHAPE_MISMATCH); seq_len may differ.
 *   out_id, out_absorbed  nullable */
cm_status cm_ingest(cm_set *set, const cm_fragment *frag, cm_stream_t stream, cm_id *out_id,
                    int32_t *out_absorbed);

/* Ingest of n deliveries in order (Algorithm 2, Ingest, applied n times): the same
 * result as n calls of cm_ingest, with one pass of GPU work for all of them (per 32
 * fragments one leaf-hash launch, which also computes the norm keys, and one or two
 * launches for the tree levels above the leaves) and a single synchronisation of
 * `stream`. A delivery whose id is
 * already in the set, or equal to an earlier delivery of the same batch, is
 * absorbed. All fragments must have the set's shape (or one common shape if the
 * set is empty). Nothing is inserted if validation fails. A delivery that fails the
 * byte check of verify_bytes_on_hit returns CM_ERR_COLLISION with the deliveries before
 * it inserted and it and the later ones not processed, as n calls of cm_ingest that
 * stop at the failing one.
 *   frags         HOST array of n descriptors (n >= 0)
 *   out_ids       nullable HOST array of n ids
 *   out_absorbed  nullable HOST array of n flags */
cm_status cm_ingest_batch(cm_set *set, const cm_fragment *frags, int32_t n, cm_stream_t stream,
                          cm_id *out_ids, int32_t *out_absorbed);

/* Ingest of n deliveries into several sets (Algorithm 2, Ingest, applied to each
 * delivery): delivery i goes into sets[i]; entries may repeat, so one call can feed
 * many serving requests. The result is that of calling cm_ingest for i = 0..n-1 in
 * order; the GPU work for all deliveries is one pass (as in cm_ingest_batch) with a
 * single synchronisation of `stream`. All sets must come from one context
 * (CM_ERR_INVALID_ARG); each delivery must have its set's shape, where a set that is
 * empty takes the shape of its first delivery (CM_ERR_SHAPE_MISMATCH). Different sets
 * may have different shapes. Nothing is inserted if validation fails; on
 * CM_ERR_COLLISION the deliveries before the failing one are inserted (as in
 * cm_ingest_batch).
 *   sets          HOST array of n set pointers
 *   frags         HOST array of n descriptors (n >= 0)
 *   out_ids       nullable HOST array of n ids
 *   out_absorbed  nullable HOST array of n flags */
cm_status cm_ingest_many(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                         cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed);

/* Merge of Algorithm 2 (Eq. setunion): dst := dst u src. Host only, no GPU work.
 * Both sets must come from the same context (CM_ERR_INVALID_ARG otherwise) and have
 * the same shape unless one is empty (CM_ERR_SHAPE_MISMATCH). On equal ids dst keeps
 * its record (the bytes are equal). dst == src is allowed (idempotent). */
cm_status cm_union(cm_set *dst, const cm_set *src);

/* Number of distinct fragments in the set. */
cm_status cm_set_size(const cm_set *set, int64_t *out);

/* Rendered length of the set: the sum of its fragments' seq_len (0 if empty). */
cm_status cm_set_seq_len(const cm_set *set, int64_t *out);

/* The set's ids in ascending order (bytes compared as a big-endian integer).
 * Writes min(size, capacity) ids to the HOST array out. */
cm_status cm_set_ids(const cm_set *set, cm_id *out, int64_t capacity);

/* Membership of ids in the set (Section 4.4: the state is the set of fragment
 * identities). out_present[i] = 1 if ids[i] is in the set, else 0. With cm_set_ids
 * this lets two replicas exchange ids first and ship only the fragments the other
 * side lacks; the union that results is the same as shipping the whole state
 * (Eq. setunion). Host only.
 *   ids, out_present  HOST arrays of n entries (n >= 0) */
cm_status cm_set_contains(const cm_set *set, const cm_id *ids, int64_t n, uint8_t *out_present);

/* The inclusion order of Section 4.4: *out = 1 if every id of a is in b (a is below
 * b in the join-semilattice), else 0. The sets may come from different contexts.
 * Host only. */
cm_status cm_set_leq(const cm_set *a, const cm_set *b, int32_t *out);

/* Render(S) of Algorithm 2 = CanonicalMerge (Algorithm 1) of the set's fragments:
 * order them by descending routing-layer mean K-norm over the last T* = min seq_len
 * positions (Eq. rho), ties by descending id; place them along the sequence axis
 * at offsets s = exclusive prefix sums of seq_len (Section 4.2); copy V; copy K of
 * the slot at offset 0; rotate every other slot's K by R(s) (Eq. bagmerge-k).
 * The kernel is enqueued on `stream` and the call returns without waiting.
 *   k_out, v_out     DEVICE, 16-byte aligned, [L][H][capacity_tokens][d] bf16
 *   capacity_tokens  must be >= the rendered length (CM_ERR_CAPACITY)
 *   out_seq_len      nullable; receives the rendered length
 *   out_order        nullable HOST array of set-size ids: the canonical order
 * The output bytes are a pure function of the set: identical for every delivery
 * order and re-delivery. An empty set renders to length 0 and launches nothing
 * (k_out and v_out may then be NULL). k_out and v_out must not overlap each other
 * or any fragment of the set (the render reads the fragments while it writes). */
cm_status cm_render(const cm_set *set, void *k_out, void *v_out, int64_t capacity_tokens,
                    cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order);

/* Ingest, Merge and Render of Algorithm 2 in one call, with the render overlapping the
 * content address where the paper's definitions allow it. The result (sets, ids,
 * absorption flags, rendered bytes, order) is that of
 *     cm_ingest_many(sets, frags, n, stream, out_ids, out_absorbed);
 *     cm_union(target, s) for every set s of `sets` other than target, in order of first
 *         appearance (the replicas' states merged into target, Eq. setunion);
 *     cm_render(target, k_out, v_out, capacity_tokens, stream, out_seq_len, out_order);
 * Overlap: the routing-layer norm keys (Eq. rho) of the deliveries are computed as the
 * call starts, beside the content address (one pass over K[l*], 1/(2L) of the bytes, and
 * a synchronisation). Byte-identical
 * fragments have equal norm keys, so members of the prospective set (the target's
 * fragments, the other sets', every delivery) whose integer tail sums S, lengths and
 * per-token norm keys all agree are taken for one fragment; if the remaining S are
 * pairwise distinct, the canonical order of Algorithm 1 does not depend on the ids: the
 * render starts at once on a stream of the context, with narrow CTAs, while the content
 * address runs on `stream`. When the ids are known the set is checked to hold exactly
 * the fragments rendered, in that order (different fragments taken for one, or sharing
 * an address, which the paper's collision assumption excludes, fail the check; then the
 * target is rendered again after the first render, so the result is still exact). With
 * a tie of S between members that differ in length or norm keys, with the re-delivery
 * fast path on, or with an output the render would refuse, the steps run one after the
 * other.
 *   sets, frags      HOST arrays of n (n >= 0): delivery i goes into sets[i]; all sets
 *                    and target from one context (CM_ERR_INVALID_ARG)
 *   target           the set rendered (it may appear in sets or not)
 *   k_out, v_out, capacity_tokens   as in cm_render
 *   out_ids, out_absorbed           nullable HOST arrays of n, as in cm_ingest_many
 *   out_seq_len, out_order          nullable, as in cm_render (out_order: the target's size)
 *   out_overlapped   nullable: 1 if the render that ran beside the content address
 *                    stood, else 0
 * The target, every other set named and every delivery must share one (L, H, d)
 * (empty sets excepted): CM_ERR_SHAPE_MISMATCH before any work otherwise. The call
 * returns after the ids reached the host; the render is then still running, ordered
 * before any later work on `stream`. On an error after the GPU work began (a collision
 * under verify_bytes_on_hit, capacity, CUDA) the sets are as the sequence above leaves
 * them at its failing step and the contents of k_out and v_out are unspecified. */
cm_status cm_ingest_render(cm_set *const *sets, const cm_fragment *frags, int32_t n,
                           cm_set *target, void *k_out, void *v_out, int64_t capacity_tokens,
                           cm_stream_t stream, cm_id *out_ids, int32_t *out_absorbed,
                           int64_t *out_seq_len, cm_id *out_order, int32_t *out_overlapped);

/* One render job of cm_render_many: a set and its contiguous output, with the
 * meaning of the arguments of the same names in cm_render. */
typedef struct cm_render_job {
    const cm_set *set;
    void *k_out;                  /* DEVICE, 16-byte aligned, [L][H][capacity_tokens][d] bf16 */
    void *v_out;
    int64_t capacity_tokens;
} cm_render_job;

/* Render(S) of Algorithm 2 for several sets in one pass: jobs[i].set is rendered
 * into jobs[i].k_out / v_out exactly as cm_render would (the same bytes), but the
 * slots of all sets are packed into shared launches of the render kernel instead
 * of at least one launch per set, which keeps the GPU full when the sets are small
 * (many concurrent serving requests). All sets must come from one context
 * (CM_ERR_INVALID_ARG) and every non-empty set must have the same (L, H, d)
 * (CM_ERR_SHAPE_MISMATCH); each job is validated as in cm_render before anything
 * is launched. Outputs must not overlap one another or any fragment of any job.
 * Enqueued on `stream`; returns without waiting.
 *   jobs          HOST array of n jobs (n >= 0)
 *   out_seq_lens  nullable HOST array of n: the rendered length of each set */
cm_status cm_render_many(const cm_render_job *jobs, int32_t n, cm_stream_t stream,
                         int64_t *out_seq_lens);

/* Incremental Render(S) (addresses the lazy O(m) re-render of Section 7): k_out and
 * v_out already hold the render of an earlier state whose canonical order was
 * prev_order[0..prev_n) (as returned by cm_render / this call). Slots of the longest
 * common prefix of that order and the set's new canonical order keep their offsets,
 * so their bytes are left in place; every later slot is rendered again from its
 * unshifted fragment (a shifted slot cannot be re-rotated from its previous render
 * without a second rounding). The result is byte-identical to cm_render into a fresh
 * buffer. The caller guarantees that the buffer holds what prev_order says (the
 * library cannot check it); prev_n = 0 is a full render.
 *   out_reused_tokens  nullable; receives the number of tokens left in place
 * Other arguments and the asynchrony are as for cm_render. */
cm_status cm_render_incremental(const cm_set *set, void *k_out, void *v_out,
                                int64_t capacity_tokens, const cm_id *prev_order, int64_t prev_n,
                                cm_stream_t stream, int64_t *out_seq_len, cm_id *out_order,
                                int64_t *out_reused_tokens);

/* A paged KV cache (PagedAttention-style block pools) as a render destination.
 * Token position pos of (layer l, kv head h) lives at element
 *   block_table[pos / block_size] * stride_block + l * stride_layer + h * stride_head
 *   + (pos % block_size) * stride_token
 * of k_pool (K) and v_pool (V); head_dim elements are contiguous from there. Strides
 * are in bf16 elements and must be multiples of 8 (16 bytes); pools 16-byte aligned.
 * This covers the usual layouts, e.g. per-layer pools [L][num_blocks][block_size][H][d]
 * or block-major [num_blocks][L][H][block_size][d]. */
typedef struct cm_paged_cache {
    void *k_pool;                 /* DEVICE */
    void *v_pool;                 /* DEVICE */
    const int32_t *block_table;   /* DEVICE: logical block -> physical block index */
    int64_t table_entries;        /* capacity = table_entries * block_size tokens */
    int64_t block_size;           /* tokens per block, >= 1 */
    int64_t stride_block;
    int64_t stride_layer;
    int64_t stride_head;
    int64_t stride_token;
} cm_paged_cache;

/* Render(S) (Algorithm 2; Algorithm 1) into a paged cache: the same bytes as cm_render,
 * each merged position written to its block (Section 4.5: the merge is compatible with
 * PagedAttention-style block-addressable caches). The physical blocks named by the first
 * ceil(rendered length / block_size) table entries must be distinct and inside the pools
 * (the table is on the device and is not checked); positions beyond the rendered length
 * are left untouched. CM_ERR_CAPACITY if the table is too short. Asynchronous on `stream`. */
cm_status cm_render_paged(const cm_set *set, const cm_paged_cache *out, cm_stream_t stream,
                          int64_t *out_seq_len, cm_id *out_order);

/* BagMerge (Section 4.2, Eq. bagmerge-k / bagmerge-v) in the caller's order:
 * frags[0] at offset 0 (byte copy), frags[i] at the sum of the previous seq_len,
 * K rotated by R(offset), V copied. No content address, no dedup: passing the same
 * fragment twice renders it twice (the naive multiset re-render of Section 5.9).
 * All fragments must share (L, H, d). Enqueued on `stream`; returns without waiting.
 *   frags  HOST array of n >= 1 descriptors;  other arguments as in cm_render */
cm_status cm_bagmerge(cm_context *ctx, const cm_fragment *frags, int32_t n, void *k_out,
                      void *v_out, int64_t capacity_tokens, cm_stream_t stream,
                      int64_t *out_seq_len);

/* Synchronise `stream` and report whether any render launched from ctx since the
 * last check had a device-side wait run out (render kernels bound every wait on
 * their own TMA copies to about one second, then record the failure and return
 * instead of hanging). Returns CM_ERR_TIMEOUT once per such event and clears it;
 * the output of the affected render is incomplete. CM_OK otherwise. */
cm_status cm_context_check(cm_context *ctx, cm_stream_t stream);

/* Re-delivery fast path for every later cm_ingest, cm_ingest_batch and cm_ingest_many
 * on ctx (off by default). The content address is a function of a fragment's bytes,
 * shapes and dtype (Section 4.3), so a delivery byte-identical to a fragment whose id is
 * known has that id without hashing it. With the path on, each delivery is first
 * compared byte for byte with at most 16 fragments of its exact shape and length: the
 * records its set holds, then the earlier deliveries of the same call (identical (k, v)
 * pointers count as equal without reading them). A delivery found equal takes that
 * fragment's id and norm key and is not hashed; the others are hashed as usual. Results
 * (ids, absorption, the set) are identical with the path on or off. The candidates'
 * first 4 KiB are compared first; only the first candidate whose prefix matches is then
 * compared in full, reading both fragments at HBM speed. This costs one more stream
 * synchronisation per call that has candidates (two if a prefix matches): turn it on
 * where re-deliveries are common (gossip, retries). The paper has no counterpart. */
cm_status cm_context_set_dedup_by_bytes(cm_context *ctx, int32_t enable);

/* Whether cm_ingest_render may run its render beside the content address (a scheduling
 * choice; the results are identical either way; the paper has no counterpart):
 *   0  never: the call runs cm_ingest_many, the unions and cm_render one after the other
 *   1  (the default) whenever the norm keys decide the canonical order on their own
 * CM_ERR_INVALID_ARG for any other value. */
cm_status cm_context_set_overlap(cm_context *ctx, int32_t mode);

/* Width of the render kernel's CTAs for every later render launched from ctx (a
 * scheduling aid; the paper has no counterpart). The render is one persistent CTA per
 * SM. warps = 16 (the default) gives it the whole register file of each SM: the fastest
 * render when it runs alone. warps = 8 leaves half of each SM's registers free, so that
 * the content-address kernels of a later cm_ingest* call on another stream run beside
 * the render instead of after it (the render is bound by HBM, hashing by the integer
 * ALU): a serving loop that renders one group of requests while hashing the next gains
 * throughput, at some cost to a render that runs alone. The rendered bytes are the same.
 * CM_ERR_INVALID_ARG for any other value. */
cm_status cm_context_set_render_warps(cm_context *ctx, int32_t warps);

/* Device time per kernel, accumulated while timing is on (a profiling aid). */
typedef struct cm_kernel_times {
    double leaf_hash_ms;          /* content address, level 0 (one launch per up to 32 fragments) */
    int64_t leaf_hash_launches;
    double inner_hash_ms;         /* content address, tree levels above the leaves (one
                                     kernel per call, or two when the call has 32,768 or
                                     more level-1 nodes: level 1, then the levels above) */
    int64_t inner_hash_launches;
    double render_ms;             /* render / BagMerge */
    int64_t render_launches;
    int64_t leaf_hash_fragments;  /* fragments hashed by those leaf-hash launches */
    int64_t aux_launches;         /* launches of the small kernels (result readback, byte
                                     comparison), counted, not timed */
} cm_kernel_times;

/* Turn kernel timing on or off for ctx. While on, every launch the context makes
 * is bracketed by two CUDA events on its stream. */
cm_status cm_context_set_timing(cm_context *ctx, int32_t enable);

/* Wait for the events of every timed launch so far, add their device times to the
 * context's totals and report the totals; reset != 0 zeroes them afterwards. */
cm_status cm_context_kernel_times(cm_context *ctx, cm_kernel_times *out, int32_t reset);

/* Integer-ALU throughput of `device`, measured with two register-only kernels (a
 * profiling aid for the roofline of the content-address kernels; the paper has no
 * counterpart): chains of three-input xors (one integer-ALU instruction each), and the
 * BLAKE2s compression function of the content address applied to register data, counted
 * as the 648 operations per 64-byte block that issue on the integer ALU pipe (10 rounds x
 * 8 G x (4 xors + 4 rotations) + 8 xors; G's additions run on the FMA pipe). Both are
 * reported in 10^12 operations per second, best of three timed launches of four full
 * waves each. Synchronous; allocates and frees a small device buffer; takes a few ms.
 * The calling thread's current device is restored on return. */
cm_status cm_measure_int_alu(int32_t device, double *xor3_tops, double *compress_tops);

/* Static name of a status code. */
const char *cm_status_string(cm_status status);

/* Thread-local text of the last error raised on this thread ("" if none). */
const char *cm_last_error_message(void);

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* CM_H_ */
