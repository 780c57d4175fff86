// Content address Id(C) (Section 4.3; Algorithm 2, Id) and the routing-layer
// norm key (Eq. rho), computed in one pass over the fragment's bytes.
//
// Id is a BLAKE2s tree hash (RFC 7693 compression function; tree parameters of
// the BLAKE2 paper, Section 2.10) of the byte stream K[0] V[0] ... K[L-1] V[L-1]:
// 1024-byte leaves (depth 0), inner nodes over 16 child digests, 16-byte
// digests, shapes and dtype in the salt, seq_len in the personalisation.
//
// Level 0 runs one thread per leaf: 16 compressions of 64-byte blocks, loaded as
// 128-bit vectors straight from the fragment buffers. The same launch computes the
// norm key with one thread per row of K[l*]: the squared norm of the key in fp64 in
// ascending element order, then the quantised norm (round-half-even of 2^20 * sqrt,
// saturated at 2^44 - 1) added into Q[t] with a 64-bit integer atomic: integer
// addition is associative, so Q does not depend on the order the atomics land in.
#include "cm_bounds.h"
#include "cm_hash_kernels.h"

#include <cstring>

#include <vector>

namespace cm {
namespace {

constexpr uint32_t kIV0 = 0x6A09E667u, kIV1 = 0xBB67AE85u, kIV2 = 0x3C6EF372u, kIV3 = 0xA54FF53Au;
constexpr uint32_t kIV4 = 0x510E527Fu, kIV5 = 0x9B05688Cu, kIV6 = 0x1F83D9ABu, kIV7 = 0x5BE0CD19u;
constexpr unsigned long long kQMax = (1ull << 44) - 1;

__device__ __forceinline__ uint32_t rotr16(uint32_t x) { return __byte_perm(x, 0, 0x1032); }
__device__ __forceinline__ uint32_t rotr8(uint32_t x) { return __byte_perm(x, 0, 0x0321); }
__device__ __forceinline__ uint32_t rotr12(uint32_t x) { return __funnelshift_r(x, x, 12); }
__device__ __forceinline__ uint32_t rotr7(uint32_t x) { return __funnelshift_r(x, x, 7); }

// a + b + x on the FMA pipe. An SM sub-partition's integer ALU pipe accepts one warp
// instruction every two cycles and must take G's four xors and four rotations; a
// three-input add left to it (one IADD3) would make that ten instructions per G. As
// two multiply-adds by a 1 the compiler cannot see through (a __constant__ it must
// load, so it cannot fold the product into an add), the sum goes to the FMA pipe,
// which the compiler already gives the two-input adds: per G, 8 ALU and 6 FMA
// instructions instead of 10 and 2. Measured on a q4b-shaped fragment: 0.326 instead
// of 0.397 ms per 604 MB; rotations moved to the FMA pipe as well (a multiply and a
// high multiply by 2^25) made it slower.
__constant__ uint32_t g_one = 1;
__device__ __forceinline__ uint32_t add3(uint32_t a, uint32_t b, uint32_t x) {
    return (a + b * g_one) + x * g_one;
}

// The G mixing function of RFC 7693, Section 3.1 (rotation distances 16, 12, 8, 7).
#define CM_G(a, b, c, d, x, y)      \
    a = add3(a, b, (x));            \
    d = rotr16(d ^ a);              \
    c = c + d;                      \
    b = rotr12(b ^ c);              \
    a = add3(a, b, (y));            \
    d = rotr8(d ^ a);               \
    c = c + d;                      \
    b = rotr7(b ^ c);

// One round: four column mixes, then four diagonal mixes, message words taken in
// the order of that round's SIGMA row (RFC 7693, Section 2.7).
#define CM_ROUND(s0, s1, s2, s3, s4, s5, s6, s7, s8, s9, s10, s11, s12, s13, s14, s15) \
    CM_G(v0, v4, v8, v12, m[s0], m[s1])                                                \
    CM_G(v1, v5, v9, v13, m[s2], m[s3])                                                \
    CM_G(v2, v6, v10, v14, m[s4], m[s5])                                               \
    CM_G(v3, v7, v11, v15, m[s6], m[s7])                                               \
    CM_G(v0, v5, v10, v15, m[s8], m[s9])                                               \
    CM_G(v1, v6, v11, v12, m[s10], m[s11])                                             \
    CM_G(v2, v7, v8, v13, m[s12], m[s13])                                              \
    CM_G(v3, v4, v9, v14, m[s14], m[s15])

// Compression function F (RFC 7693, Section 3.2), 10 rounds. t = bytes hashed
// so far including this block; the last-node flag is applied together with the
// last-block flag, on the node's final compression.
__device__ __forceinline__ void compress(uint32_t h[8], const uint32_t m[16], uint64_t t,
                                         bool last_block, bool last_node) {
    uint32_t v0 = h[0], v1 = h[1], v2 = h[2], v3 = h[3];
    uint32_t v4 = h[4], v5 = h[5], v6 = h[6], v7 = h[7];
    uint32_t v8 = kIV0, v9 = kIV1, v10 = kIV2, v11 = kIV3;
    uint32_t v12 = kIV4 ^ (uint32_t)t, v13 = kIV5 ^ (uint32_t)(t >> 32);
    uint32_t v14 = last_block ? ~kIV6 : kIV6;
    uint32_t v15 = (last_block && last_node) ? ~kIV7 : kIV7;
    CM_ROUND(0, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15)
    CM_ROUND(14, 10, 4, 8, 9, 15, 13, 6, 1, 12, 0, 2, 11, 7, 5, 3)
    CM_ROUND(11, 8, 12, 0, 5, 2, 15, 13, 10, 14, 3, 6, 7, 1, 9, 4)
    CM_ROUND(7, 9, 3, 1, 13, 12, 11, 14, 2, 6, 5, 10, 4, 0, 15, 8)
    CM_ROUND(9, 0, 5, 7, 2, 4, 10, 15, 14, 1, 11, 12, 6, 8, 3, 13)
    CM_ROUND(2, 12, 6, 10, 0, 11, 8, 3, 4, 13, 7, 5, 15, 14, 1, 9)
    CM_ROUND(12, 5, 1, 15, 14, 13, 4, 10, 0, 7, 6, 3, 9, 2, 8, 11)
    CM_ROUND(13, 11, 7, 14, 12, 1, 3, 9, 5, 0, 15, 4, 8, 6, 2, 10)
    CM_ROUND(6, 15, 14, 9, 11, 3, 0, 8, 12, 2, 13, 7, 1, 4, 10, 5)
    CM_ROUND(10, 2, 8, 4, 7, 6, 1, 5, 15, 11, 9, 14, 3, 12, 13, 0)
    h[0] ^= v0 ^ v8;
    h[1] ^= v1 ^ v9;
    h[2] ^= v2 ^ v10;
    h[3] ^= v3 ^ v11;
    h[4] ^= v4 ^ v12;
    h[5] ^= v5 ^ v13;
    h[6] ^= v6 ^ v14;
    h[7] ^= v7 ^ v15;
}

#undef CM_ROUND
#undef CM_G

// Chaining value of node (offset, depth): the base words with the 48-bit node
// offset (parameter bytes 8..13) and the node depth (byte 14) xored in.
__device__ __forceinline__ void node_init(uint32_t h[8], const TreeParams &tp, uint64_t offset,
                                          uint32_t depth) {
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = tp.h_base[i];
    h[2] ^= (uint32_t)offset;
    h[3] ^= ((uint32_t)(offset >> 32) & 0xFFFFu) | (depth << 16);
}

__device__ __forceinline__ uint4 load_nc(const uint8_t *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

__device__ __forceinline__ void store_digest(uint8_t *dst, const uint32_t h[8]) {
    *reinterpret_cast<uint4 *>(dst) = make_uint4(h[0], h[1], h[2], h[3]);
}

// Bounds-checked builds: [p, p + n) lies inside the fragment's K or V array (each
// stream_bytes / 2 long); otherwise a violation is counted.
__device__ __forceinline__ bool in_fragment(const LeafLaunch &a, const uint8_t *p, uint64_t n) {
#ifdef CM_DEBUG_BOUNDS
    const uint64_t half = a.stream_bytes / 2, x = reinterpret_cast<uint64_t>(p);
    const uint64_t k = reinterpret_cast<uint64_t>(a.k), v = reinterpret_cast<uint64_t>(a.v);
    if (n <= half && ((x >= k && x - k <= half - n) || (x >= v && x - v <= half - n))) return true;
    bounds_fail();
    return false;
#else
    (void)a;
    (void)p;
    (void)n;
    return true;
#endif
}

// fl(ss + x^2) for the 8 bf16 of one 16-byte vector, in ascending element order (x^2
// is exact in fp64, so each step is the one rounding of the sum). A normal bf16 (exponent
// field 1..254) is 2^(e-127) (1 + m/128) in magnitude; as an fp64 its exponent field is
// e + 896 and its 7 fraction bits lead the 52-bit fraction, so the high word of |x| is
// ((e << 7 | m) << 13) + (896 << 20) and the low word is 0: integer operations instead of
// a conversion on the FP64 pipe, which is the slow one on this part. A vector holding a
// zero, subnormal, infinity or NaN converts through fp32 instead.
__device__ __forceinline__ double accumulate_squares(uint4 w, double ss) {
    const uint32_t words[4] = {w.x, w.y, w.z, w.w};
    bool normal = true;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t elo = words[i] & 0x7F80u, ehi = words[i] & 0x7F800000u;
        normal = normal && elo != 0u && elo != 0x7F80u && ehi != 0u && ehi != 0x7F800000u;
    }
    if (normal) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const double lo = __hiloint2double((int)(((words[i] & 0x7FFFu) << 13) + 0x38000000u), 0);
            const double hi = __hiloint2double((int)(((words[i] >> 3) & 0x0FFFE000u) + 0x38000000u), 0);
            ss = __fma_rn(lo, lo, ss);
            ss = __fma_rn(hi, hi, ss);
        }
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const double lo = (double)__uint_as_float(words[i] << 16);
            const double hi = (double)__uint_as_float(words[i] & 0xFFFF0000u);
            ss = __fma_rn(lo, lo, ss);
            ss = __fma_rn(hi, hi, ss);
        }
    }
    return ss;
}

// Norm key of row r of K[l*] (Eq. rho; the plane is [H][T][d], so r = h*T + t): one
// thread reads the row's d/8 vectors and accumulates its squared norm, then adds the
// quantised norm into Q[t].
__device__ __forceinline__ void norm_row(const LeafLaunch &a, uint64_t r) {
    const uint8_t *row = a.k + a.norm_begin / 2 + r * a.row_bytes;   // K[l*] at stream offset 2 l* plane
    const uint32_t nvec = a.row_bytes >> 4;
    double ss = 0.0;
    for (uint32_t v = 0; v < nvec; v += 4) {
        uint4 w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (v + q < nvec)
                w[q] = CM_IN_BOUNDS(row + 16 * (v + q), 16, a.k + a.norm_begin / 2, a.plane_bytes)
                           ? load_nc(row + 16 * (v + q))
                           : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (v + q < nvec) ss = accumulate_squares(w[q], ss);
    }
    const double scaled = __dsqrt_rn(ss) * 1048576.0;     // exact scaling by 2^20
    const unsigned long long q =
        (scaled < (double)kQMax) ? __double2ull_rn(scaled) : kQMax;   // NaN saturates too
    const uint64_t t = r % a.seq_len;
    if (CM_IN_BOUNDS(a.norm_key + t, 8, a.norm_key, (uint64_t)a.seq_len * 8)) atomicAdd(a.norm_key + t, q);
}

// Cursor over the fragment's byte stream K[0] V[0] K[1] V[1] ...: every segment
// (one layer of K or of V) is plane_bytes long, a multiple of 32, so a 16-byte
// vector never straddles two segments.
struct StreamCursor {
    const uint8_t *ptr;
    uint64_t left;       // bytes left in the current segment
    uint32_t layer;
    bool in_v;
};

__device__ __forceinline__ StreamCursor cursor_at(const LeafLaunch &a, uint64_t pos) {
    StreamCursor c;
    const uint64_t two_p = 2 * a.plane_bytes;
    c.layer = (uint32_t)(pos / two_p);
    const uint64_t within = pos - (uint64_t)c.layer * two_p;
    c.in_v = within >= a.plane_bytes;
    const uint64_t seg_off = c.in_v ? within - a.plane_bytes : within;
    c.ptr = (c.in_v ? a.v : a.k) + (uint64_t)c.layer * a.plane_bytes + seg_off;
    c.left = a.plane_bytes - seg_off;
    return c;
}

__device__ __forceinline__ const uint8_t *cursor_next(const LeafLaunch &a, StreamCursor &c) {
    if (c.left == 0) {
        if (c.in_v) {
            c.in_v = false;
            ++c.layer;
        } else {
            c.in_v = true;
        }
        c.ptr = (c.in_v ? a.v : a.k) + (uint64_t)c.layer * a.plane_bytes;
        c.left = a.plane_bytes;
    }
    const uint8_t *p = c.ptr;
    c.ptr += 16;
    c.left -= 16;
    return p;
}

constexpr int kLeafThreads = kLeafBlockThreads;

__global__ void __launch_bounds__(kLeafThreads)
leaf_hash_kernel(const __grid_constant__ LeafGroup grp) {
    // the blocks after the leaf blocks compute norm keys, one thread per row of K[l*]:
    // they fill SMs that the last wave of leaf blocks leaves idle
    const uint32_t x = blockIdx.x;
    const uint32_t leaf_blocks = (uint32_t)grp.block_begin[grp.count];
    if (x >= leaf_blocks) {
        const uint32_t k = x - leaf_blocks;
        uint32_t fi = 0;
        while (fi + 1 < grp.count && k >= grp.norm_block_begin[fi + 1]) ++fi;
        const LeafLaunch &a = grp.frag[fi];
        const uint64_t r = (uint64_t)(k - grp.norm_block_begin[fi]) * kLeafThreads + threadIdx.x;
        if (r < (a.plane_bytes >> (__ffs(a.row_bytes) - 1))) norm_row(a, r);
        return;
    }
    uint32_t fi = 0;                                   // the block's fragment (uniform)
    while (fi + 1 < grp.count && x >= grp.block_begin[fi + 1]) ++fi;
    const LeafLaunch &a = grp.frag[fi];
    const uint64_t leaf = (uint64_t)(x - grp.block_begin[fi]) * kLeafThreads + threadIdx.x;
    if (leaf >= a.num_leaves) return;
    const uint64_t begin = leaf * kLeafBytes;
    const uint64_t rem = a.stream_bytes - begin;
    const uint32_t len = rem < (uint64_t)kLeafBytes ? (uint32_t)rem : (uint32_t)kLeafBytes;
    const uint32_t nblocks = (len + 63) / 64;
    const bool last_node = leaf + 1 == a.num_leaves;

    uint32_t h[8];
    node_init(h, a.tree, leaf, 0);
    StreamCursor cur = cursor_at(a, begin);

    if (len == (uint32_t)kLeafBytes && cur.left >= (uint64_t)kLeafBytes) {
        // the whole leaf lies in one K or V segment
        const uint8_t *p = cur.ptr;
        if (!in_fragment(a, p, kLeafBytes)) return;
#pragma unroll 1
        for (uint32_t b = 0; b < 16; ++b) {
            const uint4 w0 = load_nc(p + 64 * b), w1 = load_nc(p + 64 * b + 16),
                        w2 = load_nc(p + 64 * b + 32), w3 = load_nc(p + 64 * b + 48);
            const uint32_t m[16] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w,
                                    w2.x, w2.y, w2.z, w2.w, w3.x, w3.y, w3.z, w3.w};
            compress(h, m, (b + 1) * 64, b == 15, last_node);
        }
        if (CM_IN_BOUNDS(a.digests + leaf * kDigestBytes, kDigestBytes, a.digests,
                         a.num_leaves * kDigestBytes))
            store_digest(a.digests + leaf * kDigestBytes, h);
        return;
    }

    for (uint32_t b = 0; b < nblocks; ++b) {
        uint4 w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            w[q] = make_uint4(0, 0, 0, 0);
            if (b * 64 + q * 16 < len) {
                const uint8_t *ptr = cursor_next(a, cur);
                if (in_fragment(a, ptr, 16)) w[q] = load_nc(ptr);
            }
        }
        const uint32_t m[16] = {w[0].x, w[0].y, w[0].z, w[0].w, w[1].x, w[1].y, w[1].z, w[1].w,
                                w[2].x, w[2].y, w[2].z, w[2].w, w[3].x, w[3].y, w[3].z, w[3].w};
        const uint32_t end = (b + 1) * 64 < len ? (b + 1) * 64 : len;
        compress(h, m, end, b + 1 == nblocks, last_node);
    }
    if (CM_IN_BOUNDS(a.digests + leaf * kDigestBytes, kDigestBytes, a.digests,
                     a.num_leaves * kDigestBytes))
        store_digest(a.digests + leaf * kDigestBytes, h);
}

// The norm-key rows of a group alone (the blocks that follow the leaf blocks in
// leaf_hash_kernel, as their own launch): one thread per row of K[l*].
__global__ void __launch_bounds__(kLeafThreads)
norm_key_kernel(const __grid_constant__ LeafGroup grp) {
    const uint32_t k = blockIdx.x;
    uint32_t fi = 0;
    while (fi + 1 < grp.count && k >= grp.norm_block_begin[fi + 1]) ++fi;
    const LeafLaunch &a = grp.frag[fi];
    const uint64_t r = (uint64_t)(k - grp.norm_block_begin[fi]) * kLeafThreads + threadIdx.x;
    if (r < (a.plane_bytes >> (__ffs(a.row_bytes) - 1))) norm_row(a, r);
}

constexpr int kInnerThreads = 32;

__global__ void __launch_bounds__(kInnerThreads)
inner_hash_kernel(const uint8_t *__restrict__ children, uint64_t num_children,
                  uint8_t *__restrict__ out, uint64_t num_nodes, uint32_t depth,
                  const __grid_constant__ TreeParams tp) {
    const uint64_t j = (uint64_t)blockIdx.x * kInnerThreads + threadIdx.x;
    if (j >= num_nodes) return;
    const uint64_t first = j * kFanout;
    const uint64_t nc64 = num_children - first;
    const uint32_t nc = nc64 < (uint64_t)kFanout ? (uint32_t)nc64 : (uint32_t)kFanout;
    const uint32_t len = nc * kDigestBytes;
    const uint32_t nblocks = (len + 63) / 64;
    const bool last_node = j + 1 == num_nodes;
    const uint8_t *src = children + first * kDigestBytes;

    uint32_t h[8];
    node_init(h, tp, j, depth);
    for (uint32_t b = 0; b < nblocks; ++b) {
        uint4 w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t off = b * 64 + q * 16;
            w[q] = off < len && CM_IN_BOUNDS(src + off, 16, children, num_children * kDigestBytes)
                       ? load_nc(src + off)
                       : make_uint4(0, 0, 0, 0);
        }
        const uint32_t m[16] = {w[0].x, w[0].y, w[0].z, w[0].w, w[1].x, w[1].y, w[1].z, w[1].w,
                                w[2].x, w[2].y, w[2].z, w[2].w, w[3].x, w[3].y, w[3].z, w[3].w};
        const uint32_t end = (b + 1) * 64 < len ? (b + 1) * 64 : len;
        compress(h, m, end, b + 1 == nblocks, last_node);
    }
    if (CM_IN_BOUNDS(out + j * kDigestBytes, kDigestBytes, out, num_nodes * kDigestBytes))
        store_digest(out + j * kDigestBytes, h);
}

// Node j of a tree level over the digests at `children` (num_children of them): its
// 16 * min(16, num_children - 16 j) bytes, at most four 64-byte blocks, staged in the
// thread's 256-byte slice of shared memory so that one copy of the compression loop
// serves every level (the tree top runs few warps per SM; unrolled copies of the
// compression would not fit the instruction cache).
__device__ __forceinline__ void hash_node_from(uint4 *stage, uint32_t len, uint8_t *out,
                                               uint64_t j, uint64_t num_nodes, uint32_t depth,
                                               const TreeParams &tp) {
    const uint32_t nblocks = (len + 63) / 64;
    const bool last_node = j + 1 == num_nodes;
    uint32_t h[8];
    node_init(h, tp, j, depth);
#pragma unroll 1
    for (uint32_t b = 0; b < nblocks; ++b) {
        const uint4 w0 = stage[4 * b], w1 = stage[4 * b + 1], w2 = stage[4 * b + 2],
                    w3 = stage[4 * b + 3];
        const uint32_t m[16] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w,
                                w2.x, w2.y, w2.z, w2.w, w3.x, w3.y, w3.z, w3.w};
        const uint32_t end = (b + 1) * 64 < len ? (b + 1) * 64 : len;
        compress(h, m, end, b + 1 == nblocks, last_node);
    }
    if (CM_IN_BOUNDS(out + j * kDigestBytes, kDigestBytes, out, num_nodes * kDigestBytes))
        store_digest(out + j * kDigestBytes, h);
}

// Loads node j's children (zero-padded to 256 bytes) into `stage`; returns their length.
// kCoherent: the children were written by other threads of the same launch, so they
// are read through L2 (ld.global.cg) instead of the non-coherent path.
template <bool kCoherent>
__device__ __forceinline__ uint32_t stage_children(uint4 *stage, const uint8_t *children,
                                                   uint64_t num_children, uint64_t j) {
    static_assert(kFanout * kDigestBytes <= 256, "an inner node must fit four blocks");
    const uint64_t first = j * kFanout;
    const uint64_t nc64 = num_children - first;
    const uint32_t nc = nc64 < (uint64_t)kFanout ? (uint32_t)nc64 : (uint32_t)kFanout;
    const uint32_t len = nc * kDigestBytes;
    const uint4 *src = reinterpret_cast<const uint4 *>(children + first * kDigestBytes);
    uint4 w[16];
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        const bool in = (uint32_t)(q * 16) < len &&
                        CM_IN_BOUNDS(src + q, 16, children, num_children * kDigestBytes);
        w[q] = in ? (kCoherent ? __ldcg(src + q) : __ldg(src + q)) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) stage[q] = w[q];
    return len;
}

__device__ __forceinline__ uint32_t arrive_acq_rel(uint32_t *counter) {
    uint32_t old;
    asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], 1;" : "=r"(old) : "l"(counter) : "memory");
    return old;
}

constexpr int kLevel1Threads = 128;

// Level 1 of up to kMaxGroup fragments: one thread per node (node_begin: prefix sums of
// the level-1 sizes), its children read straight into registers. Every lane of a warp
// hashes a node, and with no shared memory many warps fit on an SM.
__global__ void __launch_bounds__(kLevel1Threads)
level1_kernel(const __grid_constant__ TreeTop t) {
    const uint64_t g = (uint64_t)blockIdx.x * kLevel1Threads + threadIdx.x;
    if (g >= t.node_begin[t.count]) return;
    uint32_t fi = 0;
    while (fi + 1 < t.count && g >= t.node_begin[fi + 1]) ++fi;
    const TreeTopFragment &f = t.frag[fi];
    const uint64_t j = g - t.node_begin[fi];
    const uint64_t first = j * kFanout;
    const uint64_t nc64 = f.size[0] - first;
    const uint32_t nc = nc64 < (uint64_t)kFanout ? (uint32_t)nc64 : (uint32_t)kFanout;
    const uint32_t len = nc * kDigestBytes;
    const uint32_t nblocks = (len + 63) / 64;
    const bool last_node = j + 1 == f.size[1];
    const uint8_t *src = f.level[0] + first * kDigestBytes;
    uint32_t h[8];
    node_init(h, f.tree, j, 1);
#pragma unroll 1
    for (uint32_t b = 0; b < nblocks; ++b) {
        uint4 w[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t off = b * 64 + q * 16;
            w[q] = off < len && CM_IN_BOUNDS(src + off, 16, f.level[0], f.size[0] * kDigestBytes)
                       ? load_nc(src + off)
                       : make_uint4(0, 0, 0, 0);
        }
        const uint32_t m[16] = {w[0].x, w[0].y, w[0].z, w[0].w, w[1].x, w[1].y, w[1].z, w[1].w,
                                w[2].x, w[2].y, w[2].z, w[2].w, w[3].x, w[3].y, w[3].z, w[3].w};
        const uint32_t end = (b + 1) * 64 < len ? (b + 1) * 64 : len;
        compress(h, m, end, b + 1 == nblocks, last_node);
    }
    if (CM_IN_BOUNDS(f.level[1] + j * kDigestBytes, kDigestBytes, f.level[1], f.size[1] * kDigestBytes))
        store_digest(f.level[1] + j * kDigestBytes, h);
}

// Levels kStart and up (node_begin: prefix sums of the level-kStart sizes, 0 for a
// fragment without that level): one thread per level-kStart node hashes it; then,
// level by level, the thread that completes a parent's last child hashes the parent.
template <int kStart>
__global__ void __launch_bounds__(kInnerThreads)
tree_top_kernel(const __grid_constant__ TreeTop t) {
    __shared__ uint4 stage_all[kInnerThreads][16];
    uint4 *stage = stage_all[threadIdx.x];
    const uint64_t g = (uint64_t)blockIdx.x * kInnerThreads + threadIdx.x;
    if (g >= t.node_begin[t.count]) return;
    uint32_t fi = 0;
    while (fi + 1 < t.count && g >= t.node_begin[fi + 1]) ++fi;
    const TreeTopFragment &f = t.frag[fi];
    uint64_t j = g - t.node_begin[fi];
    uint32_t len = stage_children<false>(stage, f.level[kStart - 1], f.size[kStart - 1], j);
    for (uint32_t k = kStart;; ++k) {
        hash_node_from(stage, len, f.level[k], j, f.size[k], k, f.tree);
        if (k + 1 >= f.levels) break;
        // this thread finished node j of level k; the one that finishes the last child of
        // parent j / 16 hashes the parent
        const uint64_t parent = j / kFanout;
        const uint64_t first = parent * kFanout;
        const uint64_t left = f.size[k] - first;
        const uint32_t siblings = left < (uint64_t)kFanout ? (uint32_t)left : (uint32_t)kFanout;
        // one acquire-release add: it publishes this node's digest and, for the thread
        // that counts the last sibling, makes every sibling's digest visible
        if (!CM_IN_BOUNDS(f.arrivals[k + 1] + parent, 4, f.arrivals[k + 1], f.size[k + 1] * 4))
            return;
        const uint32_t done = arrive_acq_rel(f.arrivals[k + 1] + parent) + 1;
        if (done != siblings) return;
        j = parent;
        len = stage_children<true>(stage, f.level[k], f.size[k], j);
    }
}

__global__ void compare_kernel(const uint4 *__restrict__ a, const uint4 *__restrict__ b,
                               uint64_t n, unsigned int *flag) {
    uint32_t diff = 0;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (uint64_t)gridDim.x * blockDim.x) {
        const uint4 x = __ldg(a + i), y = __ldg(b + i);
        diff |= (x.x ^ y.x) | (x.y ^ y.y) | (x.z ^ y.z) | (x.w ^ y.w);
    }
    if (__any_sync(0xFFFFFFFFu, diff != 0) && (threadIdx.x & 31) == 0) atomicOr(flag, 1u);
}

}  // namespace

CM_DEFINE_BOUNDS_READER(take_hash_bounds_violations)

int leaf_hash_blocks_per_sm() {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, leaf_hash_kernel, kLeafThreads, 0) != cudaSuccess)
        return 0;
    return n;
}

cudaError_t launch_leaf_hash_group(const LeafGroup &in, cudaStream_t stream, LeafPhases phases) {
    if (in.count > (uint32_t)kMaxLeafGroup) return cudaErrorInvalidValue;
    if (in.count == 0) return cudaSuccess;
    LeafGroup g = in;
    uint64_t norm_blocks = 0;
    for (uint32_t i = 0; i < g.count; ++i) {
        const LeafLaunch &a = g.frag[i];
        const uint64_t rows = a.row_bytes ? a.plane_bytes / a.row_bytes : 0;
        g.norm_block_begin[i] = norm_blocks;
        norm_blocks += (rows + kLeafThreads - 1) / kLeafThreads;
    }
    g.norm_block_begin[g.count] = norm_blocks;
    const uint64_t leaf_blocks = g.block_begin[g.count];
    if (leaf_blocks + norm_blocks > 0x7FFFFFFFull) return cudaErrorInvalidValue;
    // leaf blocks first, then norm-key blocks; a grid of the leaf blocks alone has no
    // norm-key block, and the norm keys alone run in their own kernel
    if (phases == LeafPhases::kNormKeys) {
        if (norm_blocks == 0) return cudaSuccess;
        norm_key_kernel<<<(unsigned)norm_blocks, kLeafThreads, 0, stream>>>(g);
        return cudaGetLastError();
    }
    const uint64_t blocks = phases == LeafPhases::kBoth ? leaf_blocks + norm_blocks : leaf_blocks;
    if (blocks == 0) return cudaSuccess;
    leaf_hash_kernel<<<(unsigned)blocks, kLeafThreads, 0, stream>>>(g);
    return cudaGetLastError();
}

cudaError_t launch_leaf_hash(const LeafLaunch &a, cudaStream_t stream) {
    LeafGroup g;
    std::memset(&g, 0, sizeof g);
    g.count = 1;
    g.block_begin[1] = (a.num_leaves + kLeafThreads - 1) / kLeafThreads;   // as the host does
    g.frag[0] = a;
    return launch_leaf_hash_group(g, stream, LeafPhases::kBoth);
}

cudaError_t launch_inner_hash(const uint8_t *children, uint64_t num_children, uint8_t *out,
                              uint64_t num_nodes, uint32_t depth, const TreeParams &tree,
                              cudaStream_t stream) {
    if (num_nodes == 0) return cudaSuccess;
    const uint64_t blocks = (num_nodes + kInnerThreads - 1) / kInnerThreads;
    inner_hash_kernel<<<(unsigned)blocks, kInnerThreads, 0, stream>>>(children, num_children, out,
                                                                    num_nodes, depth, tree);
    return cudaGetLastError();
}

int tree_top_kernels(const TreeTop &t) {
    if (t.count == 0 || t.count > (uint32_t)kMaxGroup || t.node_begin[t.count] == 0) return 0;
    if (t.node_begin[t.count] < kSplitLevel1Nodes) return 1;
    for (uint32_t i = 0; i < t.count; ++i)
        if (t.frag[i].levels >= 3) return 2;
    return 1;
}

cudaError_t launch_tree_top(const TreeTop &t, cudaStream_t stream) {
    if (t.count > (uint32_t)kMaxGroup) return cudaErrorInvalidValue;
    if (t.count == 0) return cudaSuccess;
    const uint64_t total1 = t.node_begin[t.count];
    if (total1 == 0) return cudaSuccess;
    if (total1 < kSplitLevel1Nodes) {
        // one launch from level 1: the level-2 parents are hashed by the threads that
        // finish their last child, with no second launch
        tree_top_kernel<1><<<(unsigned)((total1 + kInnerThreads - 1) / kInnerThreads),
                             kInnerThreads, 0, stream>>>(t);
        return cudaGetLastError();
    }
    level1_kernel<<<(unsigned)((total1 + kLevel1Threads - 1) / kLevel1Threads), kLevel1Threads, 0,
                    stream>>>(t);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    TreeTop u = t;   // the same fragments, counted by their level-2 nodes
    for (uint32_t i = 0; i < u.count; ++i)
        u.node_begin[i + 1] = u.node_begin[i] + (u.frag[i].levels >= 3 ? u.frag[i].size[2] : 0);
    const uint64_t total2 = u.node_begin[u.count];
    if (total2 == 0) return cudaSuccess;
    tree_top_kernel<2><<<(unsigned)((total2 + kInnerThreads - 1) / kInnerThreads), kInnerThreads,
                         0, stream>>>(u);
    return cudaGetLastError();
}

cudaError_t launch_compare(const void *a, const void *b, uint64_t bytes, unsigned int *flag,
                           cudaStream_t stream) {
    const uint64_t n = bytes / 16;
    if (n == 0) return cudaSuccess;
    uint64_t blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    compare_kernel<<<(unsigned)blocks, 256, 0, stream>>>(static_cast<const uint4 *>(a),
                                                         static_cast<const uint4 *>(b), n, flag);
    return cudaGetLastError();
}

}  // namespace cm

// ---------------------------------------------------------------- allocation-free Id(C)
//
// cm_fragment_id_static computes what cm_fragment_id computes, for callers that
// cannot allocate device memory: its scratch (the digests of every tree level
// below the root) lives in the file-scope array below, which every GPU that loads
// this library holds for the life of the process. Host code never uses the
// array's name as an address: every call looks the array's device address up with
// cudaGetSymbolAddress, with the calling thread's device current, and keeps no copy
// of it, so a device reset or another context on the device, either of which can
// move the array, never leaves a stale address in use.

namespace cm {
namespace {

constexpr uint64_t kStaticMaxLeaves = 1ull << 20;                // byte stream of at most 1 GiB
constexpr size_t kStaticScratchBytes = (17u << 20) + (256u << 10);   // 17.25 MiB
}  // namespace

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

}  // namespace cm

extern "C" cm_status cm_fragment_id_static(const cm_fragment *frag, int32_t routing_layer,
                                           cm_stream_t stream, void *id_out,
                                           uint64_t *norm_key_out) {
    using namespace cm;
    try {
        cm_status st = check_fragment(frag);
        if (st != CM_OK) return st;
        if (!id_out || !norm_key_out)
            return report_error(CM_ERR_INVALID_ARG, "id_out and norm_key_out must be device pointers");
        if ((reinterpret_cast<uintptr_t>(id_out) & 15u) != 0 ||
            (reinterpret_cast<uintptr_t>(norm_key_out) & 7u) != 0)
            return report_error(CM_ERR_ALIGNMENT,
                                "id_out must be 16-byte and norm_key_out 8-byte aligned");
        const int32_t L = frag->num_layers, H = frag->num_kv_heads, T = frag->seq_len,
                      d = frag->head_dim;
        const int32_t rl = routing_layer < 0 ? L / 2 : routing_layer;
        if (rl >= L) return report_error(CM_ERR_INVALID_ARG, "routing layer >= num_layers");
        const uint64_t plane = (uint64_t)H * T * d * 2;
        const uint64_t stream_bytes = 2ull * L * plane;
        std::vector<uint64_t> sizes{(stream_bytes + kLeafBytes - 1) / kLeafBytes};
        if (sizes[0] > kStaticMaxLeaves)
            return report_error(CM_ERR_UNSUPPORTED,
                                "cm_fragment_id_static: the fragment's K and V bytes exceed the "
                                "1 GiB that its static scratch covers; use cm_fragment_id");
        while (sizes.size() == 1 || sizes.back() > 1)
            sizes.push_back((sizes.back() + kFanout - 1) / kFanout);
        // levels below the root in the static array, each 256-byte aligned; the root
        // (the last level, one node) is written straight to id_out
        std::vector<size_t> off;
        size_t used = 0;
        for (size_t k = 0; k + 1 < sizes.size(); ++k) {
            off.push_back(used);
            used += ((size_t)sizes[k] * kDigestBytes + 255) & ~(size_t)255;
        }
        if (used > kStaticScratchBytes)
            return report_error(CM_ERR_UNSUPPORTED, "static scratch layout overflow");
        cudaError_t e = cudaSuccess;
        const cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
        void *addr = nullptr;
        e = cudaGetSymbolAddress(&addr, g_static_scratch);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
        }
        uint8_t *scratch = static_cast<uint8_t *>(addr);
        e = cudaMemsetAsync(norm_key_out, 0, (size_t)T * sizeof(uint64_t), cs);
        if (e != cudaSuccess) return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
        LeafLaunch a;
        a.k = static_cast<const uint8_t *>(frag->k);
        a.v = static_cast<const uint8_t *>(frag->v);
        a.plane_bytes = plane;
        a.stream_bytes = stream_bytes;
        a.num_leaves = sizes[0];
        a.norm_begin = 2ull * (uint64_t)rl * plane;
        a.row_bytes = (uint32_t)d * 2;
        a.seq_len = (uint32_t)T;
        a.norm_key = reinterpret_cast<unsigned long long *>(norm_key_out);
        a.digests = scratch + off[0];
        a.tree = make_tree_params(L, H, d, T);
        e = launch_leaf_hash(a, cs);
        if (e != cudaSuccess) return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
        for (size_t k = 1; k < sizes.size(); ++k) {
            uint8_t *out = (k + 1 == sizes.size()) ? static_cast<uint8_t *>(id_out) : scratch + off[k];
            e = launch_inner_hash(scratch + off[k - 1], sizes[k - 1], out, sizes[k], (uint32_t)k,
                                  a.tree, cs);
            if (e != cudaSuccess) return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
        }
        return CM_OK;
    } catch (...) {
        return report_error(CM_ERR_OOM, "host allocation failed");
    }
}

// ---------------------------------------------------------------- integer-ALU throughput
//
// Register-only kernels that measure the ceiling of the content-address kernels on the
// current GPU (a profiling aid for their roofline): chains of three-input xors, one
// integer-ALU instruction each, and the compression function above applied to register
// data with no memory traffic, counted as the 648 operations per 64-byte block that
// issue on the integer ALU pipe (10 rounds x 8 G x (4 xors + 4 rotations) + 8 xors).

namespace cm {
namespace {

__global__ void __launch_bounds__(kLeafThreads)
xor3_probe_kernel(uint32_t *out, int iters) {
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i] = tid * (2u * i + 3u);
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = a[i] ^ a[(i + 1) & 7] ^ a[(i + 3) & 7];
    }
    uint32_t x = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) x ^= a[i];
    out[tid] = x;
}

__global__ void __launch_bounds__(kLeafThreads)
compress_probe_kernel(uint32_t *out, int blocks) {
    const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t h[8], m[16];
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = tid * 2654435761u + (uint32_t)i;
#pragma unroll
    for (int i = 0; i < 16; ++i) m[i] = tid ^ ((uint32_t)i * 0x9E3779B9u);
    for (int b = 0; b < blocks; ++b) {
        compress(h, m, (uint64_t)(b + 1) * 64, false, false);
        m[0] ^= h[0];
        m[7] ^= h[3];
        m[11] ^= h[6];
    }
    out[tid] = h[0] ^ h[1] ^ h[2] ^ h[3] ^ h[4] ^ h[5] ^ h[6] ^ h[7];
}

}  // namespace
}  // namespace cm

extern "C" cm_status cm_measure_int_alu(int32_t device, double *xor3_tops, double *compress_tops) {
    using namespace cm;
    if (!xor3_tops || !compress_tops)
        return report_error(CM_ERR_INVALID_ARG, "xor3_tops and compress_tops are required");
    int prev = 0;
    cudaError_t e = cudaGetDevice(&prev);
    if (e != cudaSuccess) return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
    e = cudaSetDevice(device);
    if (e != cudaSuccess) return report_error(CM_ERR_CUDA, cudaGetErrorString(e));
    cm_status st = CM_OK;
    uint32_t *out = nullptr;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    auto check = [&](cudaError_t err) {
        if (err != cudaSuccess && st == CM_OK) st = report_error(CM_ERR_CUDA, cudaGetErrorString(err));
        return err == cudaSuccess;
    };
    int sms = 0, per_sm_x = 0, per_sm_c = 0;
    if (check(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device)) &&
        check(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_x, xor3_probe_kernel,
                                                            kLeafThreads, 0)) &&
        check(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_c, compress_probe_kernel,
                                                            kLeafThreads, 0))) {
        // four full waves of each kernel
        const int grid_x = 4 * sms * per_sm_x, grid_c = 4 * sms * per_sm_c;
        const int grid = grid_x > grid_c ? grid_x : grid_c;
        const int xor_iters = 4096, comp_blocks = 64;
        if (check(cudaMalloc(&out, (size_t)grid * kLeafThreads * sizeof(uint32_t))) &&
            check(cudaEventCreate(&e0)) && check(cudaEventCreate(&e1))) {
            auto best_ms = [&](auto launch) {
                float best = 0.0f;
                for (int rep = 0; rep < 4 && st == CM_OK; ++rep) {   // rep 0 warms up
                    check(cudaEventRecord(e0));
                    launch();
                    check(cudaGetLastError());
                    check(cudaEventRecord(e1));
                    float ms = 0.0f;
                    if (check(cudaEventSynchronize(e1)) && check(cudaEventElapsedTime(&ms, e0, e1)) &&
                        rep > 0 && (best == 0.0f || ms < best))
                        best = ms;
                }
                return (double)best;
            };
            const double ms_x = best_ms([&] {
                xor3_probe_kernel<<<grid_x, kLeafThreads>>>(out, xor_iters);
            });
            const double ms_c = best_ms([&] {
                compress_probe_kernel<<<grid_c, kLeafThreads>>>(out, comp_blocks);
            });
            if (st == CM_OK) {
                const double ops_x = (double)grid_x * kLeafThreads * xor_iters * 8;
                const double ops_c = (double)grid_c * kLeafThreads * comp_blocks * 648;
                *xor3_tops = ops_x / (ms_x * 1e-3) / 1e12;
                *compress_tops = ops_c / (ms_c * 1e-3) / 1e12;
            }
        }
    }
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    if (out) cudaFree(out);
    cudaSetDevice(prev);
    return st;
}
