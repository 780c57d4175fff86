// Render: BagMerge with RoPE re-encoding (Section 4.2, Eq. bagmerge-k /
// bagmerge-v) in a given slot order; CanonicalMerge (Algorithm 1) is this with
// the canonical order computed on the host.
//
// Every (slot, layer, head) plane of K and of V is a contiguous run of T rows of
// head_dim bf16 in the source and a contiguous run at row offset s of the output
// plane, so the render is a set of streaming copies. V and the K of the slot at
// offset 0 are copied as bytes. Every other K row is rotated by R(s): the stored
// key is R(t) k, and R(s) R(0)^-1 R(t) k = R(s + t) k, so a slot's whole K is
// turned by one constant angle a_j = s * theta^(-2j/d) per frequency j (the delta
// formula of Section 2.3), pairing element j with element j + d/2.
//
// Two kernels move the items. The full-SM render (render_reg_kernel, the default) has
// every warp take one (K, V) pair of 1 KiB items at a time: its lanes load both items
// as 16-byte vectors straight into registers, rotate the K rows, and store both with
// streaming stores; 24 warps per SM keep about 48 KiB of loads in flight, where HBM
// serves this mix of reads and writes best (more bytes in flight made the same copy
// slower). The half-SM render (render_kernel, cm_context_set_render_warps(8)) runs one
// 8-warp CTA per SM that leaves half of the register file to kernels of other
// streams; its warps keep three 4 KiB items in flight each as 1-D TMA bulk copies
// into shared memory, which needs fewer warps for the same bytes in flight. For a
// rotated K item a lane takes vector v of a row's first half and vector v of its
// second half: 8 (x, y) pairs that share the lane's 8 (cos, sin) values. A render that
// runs beside the content address (cm_ingest_render) takes a narrower width still: the
// TMA kernel with one CTA of 4 warps and 6 stages per SM for large renders, the register
// kernel with one 8-warp CTA per SM for small ones (see RenderWidth).
//
// Rounding. The result must equal round-to-nearest-even-bf16 of
// fl64(fl64(x c) - fl64(y s)) (and fl64(fl64(y c) + fl64(x s))), c and s the fp64
// cosine and sine. The fast path computes z in fp32 with one fma from c and s
// rounded to fp32 and bounds its distance to the fp64 value by one bound for both
// outputs of an element pair, E = k_j (|x| + |y|) + 2^-145 with a per-frequency constant
// k_j = (1 + 2^-8) 2^-24 max(2|c|, 3|s|) (see bound_scale). If z - E and z + E (rounded
// outward) round to the same bf16, every value between them does (rounding is
// monotone), the fp64 value included, and z's rounding is the answer. Otherwise (about
// one element in five thousand) a second
// fp32 level with error-free products and a ~2^-36 bound decides, and the few it
// cannot certify are recomputed in fp64 with the operation sequence of the
// definition and rounded directly to bf16 (fp64 throughput is very low on this part,
// so it must stay rare). The output is bit-exact either way.
#include "cm_bounds.h"
#include "cm_render_kernels.h"

#include <algorithm>

namespace cm {
namespace {

static_assert(sizeof(RenderParams) <= 32764, "render parameters exceed the kernel parameter limit");

__device__ __forceinline__ void st_stream(uint4 *p, const uint4 &v) { __stcs(p, v); }

// Two fp32 -> bf16 round-to-nearest-even, `lo` in bits 0..15, `hi` in bits 16..31.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// fp64 -> bf16 bits, round to nearest, ties to even, with bf16 subnormals and
// overflow to infinity; NaN -> 0x7FC0.
__device__ uint32_t f64_to_bf16_bits(double z) {
    const unsigned long long u = (unsigned long long)__double_as_longlong(z);
    const uint32_t sign = (uint32_t)(u >> 48) & 0x8000u;
    const unsigned long long mag = u & 0x7FFFFFFFFFFFFFFFull;
    if (mag > 0x7FF0000000000000ull) return 0x7FC0u;
    if (mag == 0x7FF0000000000000ull) return sign | 0x7F80u;
    const double a = __longlong_as_double((long long)mag);
    if (a < 0x1p-126) {
        // spacing 2^-133 below the normal range; the count 128 is the smallest normal
        return sign | (uint32_t)rint(a * 0x1p133);
    }
    // keep 7 of the 52 stored significand bits: add half an ulp minus one, plus
    // the kept lsb (ties to even); a carry moves into the exponent field
    const unsigned long long r = (mag + 0x00000FFFFFFFFFFFull + ((mag >> 45) & 1ull)) >> 45;
    const int e = (int)(r >> 7) - 1023 + 127;
    if (e >= 255) return sign | 0x7F80u;
    return sign | ((uint32_t)e << 7) | (uint32_t)(r & 0x7Fu);
}

// First-level error bound. With w = fl(y s32) and z = fl(x c32 - w) (one fma),
// c32 = fl(c1 + c2) within u|c32| + 2^-40 |c| (+2^-150 if subnormal) of c, u = 2^-24:
//   |z - (x c - y s)| <= u |z| + u |x||c32| + u |w| + u |y||s32| (+ tiny terms)
//                     <= (1 + 2^-9) u (|z| + |x||c32| + 2 |y||s32|) + 2^-148 (|x| + |y|) + 2^-146,
// the last two terms covering roundings in the subnormal range (absolute error 2^-150
// each) and the fp64 value's own distance to x c - y s (below 2^-52 of the products).
// With M = max(2|c32|, 3|s32|): |z| <= (1 + u)|x||c32| + (1 + u)^2 |y||s32| + 2^-148, so
// |z| + |x||c32| + 2|y||s32| <= (1 + u) M (|x| + |y|) + 2^-148; and M >= 6/sqrt(13) > 1.66
// (c32^2 + s32^2 is within 2^-22 of 1), so 2^-148 (|x| + |y|) is far below the margin
// (2^-8 - 2^-9 - u - 2^-33) u M (|x| + |y|). Hence
//   |z - X| <= (1 + 2^-8) u M (|x| + |y|) + 2^-145 = k (|x| + |y|) + 2^-145,
// X the fp64 value, and the same for y' = fl(y c32 + fl(x s32)) (|x| and |y| swap roles,
// M stays). bound_scale returns k rounded up, from the fp32 (c32, s32) of one frequency.
__device__ __forceinline__ float bound_scale(float c32, float s32) {
    const float m = fmaxf(2.0f * fabsf(c32), __fmul_ru(3.0f, fabsf(s32)));
    return __fmul_ru(m, 0x1.01p-24f);
}

// Paired fp32 arithmetic (sm_100 and later): two fp32 operations, elementwise, in one
// instruction on a register pair; the rounding of each half is that of the scalar op.
__device__ __forceinline__ uint64_t f32x2_of(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void halves(uint64_t v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t mul2_rn(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t fma2_rn(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t sub2_rd(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("sub.rm.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t add2_ru(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rp.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
// the two halves of a pair as bf16, round to nearest even (lo in bits 0..15)
__device__ __forceinline__ uint32_t pack_pair(uint64_t v) {
    float lo, hi;
    halves(v, lo, hi);
    return pack_bf16x2(lo, hi);
}

// Rotate the pairs (x0, y0), (x1, y1) held in word xw (x0 low, x1 high) and word yw
// (frequency of pair e: c_e, s_e, ns_e = -s_e and bound scale k_e), the two pairs of a
// word in paired instructions: x' = fma(x, c, fl(y ns)), y' = fma(y, c, fl(x s)), the
// scalar operations of the bound's proof. Returns the rotated words and a mask whose
// nonzero 16-bit halves mark elements whose fp32 result is not certified. A certified
// half's z - E, z and z + E round to the same bf16 (rounding is monotone), so the
// rounding of z + E is the output there; uncertified halves are replaced by the fix-up.
__device__ __forceinline__ void rotate_word(uint32_t xw, uint32_t yw, float c0, float s0,
                                            float ns0, float k0, float c1, float s1, float ns1,
                                            float k1, uint32_t &xo, uint32_t &yo, uint32_t &bad) {
    const float x0 = bf16_lo(xw), x1 = bf16_hi(xw);
    const float y0 = bf16_lo(yw), y1 = bf16_hi(yw);
    const uint64_t X = f32x2_of(x0, x1), Y = f32x2_of(y0, y1), C = f32x2_of(c0, c1);
    const uint64_t ZX = fma2_rn(X, C, mul2_rn(Y, f32x2_of(ns0, ns1)));
    const uint64_t ZY = fma2_rn(Y, C, mul2_rn(X, f32x2_of(s0, s1)));
    // one bound for both outputs of a pair: E = k (|x| + |y|) + 2^-145, rounded up
    const uint64_t E = f32x2_of(__fmaf_ru(__fadd_ru(fabsf(x0), fabsf(y0)), k0, 0x1p-145f),
                               __fmaf_ru(__fadd_ru(fabsf(x1), fabsf(y1)), k1, 0x1p-145f));
    xo = pack_pair(add2_ru(ZX, E));
    yo = pack_pair(add2_ru(ZY, E));
    bad = (pack_pair(sub2_rd(ZX, E)) ^ xo) | (pack_pair(sub2_rd(ZY, E)) ^ yo);
}

// Second level for one element pair (x, y) whose first-level result was not
// certified. The table holds c = c1 + c2 with c1 carrying 16 significant bits
// (so x c1 and y s1 are exact fp32 products of bf16 inputs) and c2 = fp32(c - c1):
//   D = fl(x c1 - y s1),  r = fl(x c2 - fl(y s2)),  z = fl(D + r),
// within E = 2^-22 |z| + 2^-36 (|x| + |y|) + 2^-146 of the fp64 value. Certified
// as in the first level, else (rarely) recomputed in fp64 with the operation
// sequence of the definition. Returns x' in bits 0..15 and y' in bits 16..31.
__device__ __noinline__ uint32_t fix_element(float x, float y, float4 t, double c, double s) {
    const float dx = __fmaf_rn(x, t.x, -__fmul_rn(y, t.z));
    const float rx = __fmaf_rn(x, t.y, -__fmul_rn(y, t.w));
    const float zx = __fadd_rn(dx, rx);
    const float dy = __fmaf_rn(y, t.x, __fmul_rn(x, t.z));
    const float ry = __fmaf_rn(y, t.y, __fmul_rn(x, t.w));
    const float zy = __fadd_rn(dy, ry);
    const float m = __fmul_ru(__fadd_ru(fabsf(x), fabsf(y)), 0x1p-36f);
    const float ex = __fmaf_ru(fabsf(zx), 0x1p-22f, __fadd_ru(m, 0x1p-146f));
    const float ey = __fmaf_ru(fabsf(zy), 0x1p-22f, __fadd_ru(m, 0x1p-146f));
    const uint32_t lo = pack_bf16x2(__fsub_rd(zx, ex), __fsub_rd(zy, ey));
    const uint32_t hi = pack_bf16x2(__fadd_ru(zx, ex), __fadd_ru(zy, ey));
    uint32_t out = pack_bf16x2(zx, zy);
    if ((lo ^ hi) != 0u) {
        const double xd = (double)x, yd = (double)y;
        const uint32_t bx = f64_to_bf16_bits(__dsub_rn(__dmul_rn(xd, c), __dmul_rn(yd, s)));
        const uint32_t by = f64_to_bf16_bits(__dadd_rn(__dmul_rn(yd, c), __dmul_rn(xd, s)));
        out = bx | (by << 16);
    }
    return out;
}

__device__ __forceinline__ uint32_t pick_word(const uint4 &v, int w) {
    return w == 0 ? v.x : w == 1 ? v.y : w == 2 ? v.z : v.w;
}

__device__ __forceinline__ void put_half(uint4 &v, int e, uint32_t bits) {
    const int w = e >> 1;
    const uint32_t keep = (e & 1) ? 0x0000FFFFu : 0xFFFF0000u;
    const uint32_t val = (e & 1) ? (bits << 16) : bits;
    if (w == 0) v.x = (v.x & keep) | val;
    else if (w == 1) v.y = (v.y & keep) | val;
    else if (w == 2) v.z = (v.z & keep) | val;
    else v.w = (v.w & keep) | val;
}

// Re-evaluates the elements of one vector pair whose masks b0..b3 flag them. Inlined: as a
// called function its call (argument and result registers, a stack frame) cost the
// full-SM render 0.80 instead of 0.754 ms on the Qwen3-4B-shaped merge, though only about
// one warp iteration in twenty takes it.
__device__ __forceinline__ void fixup_pair(const RenderParams &p, const float4 *tab, int cs_index,
                                        const uint4 &a, const uint4 &b, uint32_t b0, uint32_t b1,
                                        uint32_t b2, uint32_t b3, uint4 &ao, uint4 &bo) {
    const uint32_t bw[4] = {b0, b1, b2, b3};
    for (int e = 0; e < 8; ++e) {
        const uint32_t m = bw[e >> 1] >> ((e & 1) * 16);
        if ((m & 0xFFFFu) == 0u) continue;
        const uint32_t xw = pick_word(a, e >> 1), yw = pick_word(b, e >> 1);
        const float x = (e & 1) ? bf16_hi(xw) : bf16_lo(xw);
        const float y = (e & 1) ? bf16_hi(yw) : bf16_lo(yw);
        const uint32_t r = fix_element(x, y, tab[cs_index + e], p.cs[2 * (cs_index + e)],
                                       p.cs[2 * (cs_index + e) + 1]);
        put_half(ao, e, r & 0xFFFFu);
        put_half(bo, e, r >> 16);
    }
}

// ---------------------------------------------------------------- TMA bulk pipeline

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Waits for phase `parity` of an mbarrier for at most kWaitLimitNs; false on timeout.
constexpr uint64_t kWaitLimitNs = 1000000000ull;
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > kWaitLimitNs) return false;
    }
    return true;
}

// 1-D bulk copy global -> shared, completion counted in bytes on `bar`.
__device__ __forceinline__ void bulk_load(void *dst_smem, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_addr(dst_smem)), "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

constexpr int kStagesDefault = 3;                   // per warp
constexpr uint32_t kItemBytes = 4096;               // one work item = one stage
// Per frequency: (c1, c2, s1, s2), then the first-level bound scale k, -s32, c32 and s32
// (one array of kMaxTablePairs each), so that an item's 8 fp32 (cos, sin) are 4 loads
constexpr size_t kTableBytes = (sizeof(float4) + 4 * sizeof(float)) * kMaxTablePairs;
// Dynamic shared memory of a CTA of kW warps: the warps' stages, then the (cos, sin) table.
template <int kW, int kStages = kStagesDefault>
constexpr size_t dyn_smem() { return (size_t)kW * kStages * kItemBytes + kTableBytes; }

// One work item: up to kItemBytes of one source plane and where it goes.
struct Item {
    const uint8_t *src;
    uint8_t *dst;        // contiguous: first output row; paged: pool + (layer, head) offset
    int64_t pos0;        // output position of the first row (paged outputs)
    uint32_t bytes;
    int32_t rows;
    int32_t rotate;      // 1: K of a slot at a nonzero offset
    int32_t cs_index;    // first (cos, sin) of this slot
#ifdef CM_DEBUG_BOUNDS
    const uint8_t *src_base;   // the slot's K or V fragment
    uint64_t src_size;
    const uint8_t *dst_base;   // the slot's K or V output (paged: the pool, whose size the
    uint64_t dst_size;         // library is not told: only the lower end is checked)
#endif
};

// Physical block of logical block b of a paged output (in bounds-checked builds: an index
// outside the table or a negative entry counts a violation and reads as block 0).
__device__ __forceinline__ int64_t table_entry(const RenderParams &p, int64_t b) {
#ifdef CM_DEBUG_BOUNDS
    if (b < 0 || !CM_IN_BOUNDS(p.block_table + b, 4, p.block_table, (uint64_t)p.table_entries * 4)) {
        if (b < 0) bounds_fail();
        return 0;
    }
    const int64_t blk = __ldg(p.block_table + b);
    if (blk < 0) {
        bounds_fail();
        return 0;
    }
    return blk;
#else
    return __ldg(p.block_table + b);
#endif
}

// Paged outputs: where the rows of one item go. When the block size is a power of two
// no smaller than the item's row count, the item's positions lie in at most two logical
// blocks: rows [0, split) in the first at a + r * stride, the rest in the next at
// b + r * stride (b is offset back by split rows so that one formula serves both), and
// the block table is read once per item instead of once per row.
struct PagedRows {
    uint8_t *a;
    uint8_t *b;
    int64_t stride;  // bytes between consecutive positions of a block
    int split;       // rows in the item's first block
    bool fast;
};

__device__ __forceinline__ PagedRows paged_rows(const RenderParams &p, const Item &it) {
    PagedRows pr;
    pr.fast = p.log2_block_size >= 0 && (int64_t)it.rows <= p.block_size;
    pr.a = pr.b = it.dst;
    pr.stride = p.stride_token * 2;
    pr.split = it.rows;
    if (pr.fast) {
        const int64_t b0 = it.pos0 >> p.log2_block_size;
        const int64_t o0 = it.pos0 & (p.block_size - 1);
        const int64_t k = p.block_size - o0;                 // rows left in block b0
        pr.a = it.dst + table_entry(p, b0) * p.stride_block * 2 + o0 * pr.stride;
        if (k < it.rows) {
            pr.split = (int)k;
            pr.b = it.dst + table_entry(p, b0 + 1) * p.stride_block * 2 - k * pr.stride;
        }
    }
    return pr;
}

// Start of output row r of an item: contiguous rows, or the row's slot in its block.
template <bool kPaged>
__device__ __forceinline__ uint4 *row_dst(const RenderParams &p, const Item &it, int r,
                                          const PagedRows &pr) {
    if (!kPaged) return reinterpret_cast<uint4 *>(it.dst) + (int64_t)r * (p.head_dim >> 3);
    if (pr.fast) return reinterpret_cast<uint4 *>((r < pr.split ? pr.a : pr.b) + (int64_t)r * pr.stride);
    const int64_t pos = it.pos0 + r;
    int64_t b, o;
    if (p.log2_block_size >= 0) {                       // the usual case: shifts
        b = pos >> p.log2_block_size;
        o = pos & ((1ll << p.log2_block_size) - 1);
    } else if (pos < 0x80000000ll && p.block_size < 0x80000000ll) {   // 32-bit division
        const uint32_t q = (uint32_t)pos / (uint32_t)p.block_size;
        b = q;
        o = pos - (int64_t)q * p.block_size;
    } else {
        b = pos / p.block_size;
        o = pos - b * p.block_size;
    }
    const int64_t blk = table_entry(p, b);
    return reinterpret_cast<uint4 *>(it.dst + (blk * p.stride_block + o * p.stride_token) * 2);
}

// Byte copy of one staged item: shared memory -> registers -> 16-byte streaming stores.
template <bool kPaged>
__device__ __forceinline__ void copy_from_smem(const RenderParams &p, const Item &it,
                                               const uint8_t *buf, int lane) {
    constexpr int kU = kItemBytes / 16 / 32;          // 8 vectors per lane
    const int n_vec = (int)(it.bytes >> 4);
    const uint4 *src = reinterpret_cast<const uint4 *>(buf);
    PagedRows pr{};
    if (kPaged) pr = paged_rows(p, it);
    uint4 r[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u)
        if (lane + 32 * u < n_vec) r[u] = src[lane + 32 * u];
    if (!kPaged) {
        uint4 *dst = reinterpret_cast<uint4 *>(it.dst);
#pragma unroll
        for (int u = 0; u < kU; ++u)
            if (lane + 32 * u < n_vec && CM_IN_BOUNDS(dst + lane + 32 * u, 16, it.dst_base, it.dst_size))
                st_stream(dst + lane + 32 * u, r[u]);
    } else {
        const int log2_vpr = p.log2_pairs_per_row + 1;     // vectors per row = d / 8
        const int col_mask = (1 << log2_vpr) - 1;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int v = lane + 32 * u;
            if (v < n_vec) {
                uint4 *q = row_dst<true>(p, it, v >> log2_vpr, pr) + (v & col_mask);
                if (CM_IN_BOUNDS(q, 16, it.dst_base, it.dst_size)) st_stream(q, r[u]);
            }
        }
    }
}

// K rows of one staged item: rotate and store. Lane `lane` takes vector pairs
// q = lane, lane + 32, ...; its vector index within the row half is lane % (d/16),
// the same for every q, so its 8 (cos, sin) values are loaded once per item.
template <bool kPaged>
__device__ __forceinline__ void rotate_from_smem(const RenderParams &p, const float4 *tab,
                                                 const float *kt, const float *nst, const float *c32,
                                                 const float *s32, const Item &it,
                                                 const uint8_t *buf, int lane, int lane_v) {
    const int vecs_per_row = p.head_dim >> 3;
    const int half_vecs = p.head_dim >> 4;
    const int n_pairs = it.rows * half_vecs;
    const int cs_index = it.cs_index + 8 * lane_v;
    PagedRows pr{};
    if (kPaged) pr = paged_rows(p, it);
    float c[8], s[8];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const float4 cv = *reinterpret_cast<const float4 *>(c32 + cs_index + 4 * h);
        const float4 sv = *reinterpret_cast<const float4 *>(s32 + cs_index + 4 * h);
        c[4 * h] = cv.x, c[4 * h + 1] = cv.y, c[4 * h + 2] = cv.z, c[4 * h + 3] = cv.w;
        s[4 * h] = sv.x, s[4 * h + 1] = sv.y, s[4 * h + 2] = sv.z, s[4 * h + 3] = sv.w;
    }
    const uint4 *src = reinterpret_cast<const uint4 *>(buf);
#pragma unroll 1
    for (int q = lane; q < n_pairs; q += 32) {
        const int row = q >> p.log2_pairs_per_row;
        const int off = row * vecs_per_row + lane_v;
        const uint4 a = src[off];
        const uint4 b = src[off + half_vecs];
        const float4 ka = *reinterpret_cast<const float4 *>(kt + cs_index);
        const float4 kb = *reinterpret_cast<const float4 *>(kt + cs_index + 4);
        const float4 na = *reinterpret_cast<const float4 *>(nst + cs_index);
        const float4 nb = *reinterpret_cast<const float4 *>(nst + cs_index + 4);
        uint4 ao, bo;
        uint32_t b0, b1, b2, b3;
        rotate_word(a.x, b.x, c[0], s[0], na.x, ka.x, c[1], s[1], na.y, ka.y, ao.x, bo.x, b0);
        rotate_word(a.y, b.y, c[2], s[2], na.z, ka.z, c[3], s[3], na.w, ka.w, ao.y, bo.y, b1);
        rotate_word(a.z, b.z, c[4], s[4], nb.x, kb.x, c[5], s[5], nb.y, kb.y, ao.z, bo.z, b2);
        rotate_word(a.w, b.w, c[6], s[6], nb.z, kb.z, c[7], s[7], nb.w, kb.w, ao.w, bo.w, b3);
        if ((b0 | b1 | b2 | b3) != 0u) fixup_pair(p, tab, cs_index, a, b, b0, b1, b2, b3, ao, bo);
        uint4 *d = row_dst<kPaged>(p, it, row, pr) + lane_v;
        if (CM_IN_BOUNDS(d, 16, it.dst_base, it.dst_size)) st_stream(d, ao);
        if (CM_IN_BOUNDS(d + half_vecs, 16, it.dst_base, it.dst_size)) st_stream(d + half_vecs, bo);
    }
}

// (c1, c2) split of an fp64 cosine or sine: c1 = fp32(c) with its low 8 significand
// bits cleared (16 significant bits), c2 = fp32(c - c1).
__device__ __forceinline__ float2 split16(double c) {
    const float c1 = __uint_as_float(__float_as_uint(__double2float_rn(c)) & 0xFFFFFF00u);
    return make_float2(c1, __double2float_rn(c - (double)c1));
}

// A (K, V) item pair: the same rows of one (slot, layer, head) plane of K and of V.
struct Pair {
    const uint8_t *ks, *vs;   // sources
    uint8_t *kd, *vd;         // contiguous: first output row; paged: pool + (layer, head) offset
    int64_t pos0;             // output position of the first row
    int32_t rows;
    int32_t rotate;
    int32_t cs_index;
#ifdef CM_DEBUG_BOUNDS
    const uint8_t *ks_base, *vs_base, *kd_base, *vd_base;
    uint64_t src_size, dst_size;
#endif
};

// The pairs pr = first, first + stride, ... of a warp. Pair pr of a launch is pair
// pr - chunk_begin / 2 of its slot: row chunk c of (layer, head) plane lhp. Along the
// stride, (plane, chunk) advance by additions; only entering a slot costs a search
// and a division.
struct PairWalk {
    uint32_t pr, npairs, stride;
    int si;
    uint32_t lhp, c, st_l, st_c;
    uint32_t l, h, st_pl, st_ph;   // paged outputs: lhp = l * H + h, st_l = st_pl * H + st_ph

    template <bool kPaged>
    __device__ __forceinline__ void enter(const RenderParams &p) {
        si = 0;
        while (si + 1 < p.num_slots && 2 * pr >= p.slot[si + 1].chunk_begin) ++si;
        const RenderSlot &S = p.slot[si];
        const uint32_t local = pr - (S.chunk_begin >> 1);
        lhp = local / S.chunks_per_plane;
        c = local - lhp * S.chunks_per_plane;
        st_l = stride / S.chunks_per_plane;
        st_c = stride - st_l * S.chunks_per_plane;
        if (kPaged) {
            const uint32_t H = (uint32_t)p.num_heads;
            l = lhp / H;
            h = lhp - l * H;
            st_pl = st_l / H;
            st_ph = st_l - st_pl * H;
        }
    }
    template <bool kPaged>
    __device__ __forceinline__ bool next(const RenderParams &p) {
        pr += stride;
        if (pr >= npairs) return false;
        const uint32_t cpp = p.slot[si].chunks_per_plane;
        c += st_c;
        lhp += st_l;
        uint32_t carry = 0;
        if (c >= cpp) {
            c -= cpp;
            ++lhp;
            carry = 1;
        }
        if (lhp >= (uint32_t)(p.num_layers * p.num_heads)) {
            enter<kPaged>(p);
        } else if (kPaged) {
            const uint32_t H = (uint32_t)p.num_heads;
            h += st_ph + carry;   // < 2H: one correction
            l += st_pl;
            if (h >= H) {
                h -= H;
                ++l;
            }
        }
        return true;
    }
};

template <bool kPaged>
__device__ __forceinline__ Pair pair_of(const RenderParams &p, const PairWalk &w) {
    const RenderSlot &S = p.slot[w.si];
    const int64_t row_bytes = (int64_t)p.head_dim * 2;
    const int64_t row0 = (int64_t)w.c * p.rows_per_chunk;
    const int64_t left = S.seq_len - row0;
    Pair q;
    q.rows = left < p.rows_per_chunk ? (int)left : p.rows_per_chunk;
    const int64_t so = ((int64_t)w.lhp * S.seq_len + row0) * row_bytes;
    q.ks = static_cast<const uint8_t *>(S.k) + so;
    q.vs = static_cast<const uint8_t *>(S.v) + so;
    if (kPaged) {
        const int64_t o = ((int64_t)w.l * p.stride_layer + (int64_t)w.h * p.stride_head) * 2;
        q.kd = static_cast<uint8_t *>(p.k_pool) + o;
        q.vd = static_cast<uint8_t *>(p.v_pool) + o;
    } else {
        const int64_t o = ((int64_t)w.lhp * S.capacity + S.offset + row0) * row_bytes;
        q.kd = static_cast<uint8_t *>(S.k_out) + o;
        q.vd = static_cast<uint8_t *>(S.v_out) + o;
    }
    q.pos0 = S.offset + row0;
    q.rotate = S.rotate;
    q.cs_index = S.table_base;
#ifdef CM_DEBUG_BOUNDS
    const uint64_t lh_planes = (uint64_t)p.num_layers * (uint64_t)p.num_heads;
    q.ks_base = static_cast<const uint8_t *>(S.k);
    q.vs_base = static_cast<const uint8_t *>(S.v);
    q.src_size = lh_planes * (uint64_t)S.seq_len * (uint64_t)row_bytes;
    if (p.paged) {
        q.kd_base = static_cast<const uint8_t *>(p.k_pool);
        q.vd_base = static_cast<const uint8_t *>(p.v_pool);
        q.dst_size = ~0ull - reinterpret_cast<uint64_t>(q.kd_base > q.vd_base ? q.kd_base : q.vd_base);
    } else {
        q.kd_base = static_cast<const uint8_t *>(S.k_out);
        q.vd_base = static_cast<const uint8_t *>(S.v_out);
        q.dst_size = lh_planes * (uint64_t)S.capacity * (uint64_t)row_bytes;
    }
#endif
    return q;
}

// The K or V half of a pair as an Item (for the placement helpers).
__device__ __forceinline__ Item half_item(const Pair &q, bool v) {
    Item it;
    it.src = v ? q.vs : q.ks;
    it.dst = v ? q.vd : q.kd;
    it.pos0 = q.pos0;
    it.rows = q.rows;
    it.bytes = 0;
    it.rotate = v ? 0 : q.rotate;
    it.cs_index = q.cs_index;
#ifdef CM_DEBUG_BOUNDS
    it.src_base = v ? q.vs_base : q.ks_base;
    it.src_size = q.src_size;
    it.dst_base = v ? q.vd_base : q.kd_base;
    it.dst_size = q.dst_size;
#endif
    return it;
}

// Half-SM render: a persistent kernel with one CTA of kW = 8 warps per SM (half of the
// register file, leaving room for kernels of other streams on the same SMs; kW = 4 with 6
// stages beside the leaf hash); every warp runs its own pipeline over its own items, with
// no block-wide barrier after set-up. Items come in (K, V) pairs of the same (slot, layer,
// head, row chunk); a warp takes pairs warp id + m * total warps and does the K item,
// then the V item, so rotation work and pure copies alternate within every warp. Lane 0
// keeps up to kStages items in flight as 1-D TMA bulk loads into the warp's stages
// (completion on one mbarrier per stage); all lanes wait for an item, move it from shared
// memory to its place in the output (rotating K rows of slots at a nonzero offset; kPaged:
// each row's place comes from the block table), and lane 0 refills the stage with the
// warp's next item. Every wait is bounded: on timeout the warp records an error, waits
// (bounded) for its own copies in flight and returns.
template <bool kPaged, int kW, int kStages = kStagesDefault, int kMinBlocks = 16 / kW>
__global__ void __launch_bounds__(kW * 32, kMinBlocks)
render_kernel(const __grid_constant__ RenderParams p) {
    constexpr int kThreads = kW * 32;
    extern __shared__ __align__(128) uint8_t smem[];
    // item j of a warp: its data in stage j % kStages, its Item in entry j % kRing (one
    // entry more than stages, so that a pair's V Item can be written with its K Item)
    constexpr int kRing = kStages + 1;
    __shared__ __align__(8) uint64_t full[kW][kStages];
    __shared__ Item items[kW][kRing];
    __shared__ PairWalk walks[kW];   // lane 0's position along its warp's pairs
    float4 *tab = reinterpret_cast<float4 *>(smem + (size_t)kW * kStages * kItemBytes);
    float *kt = reinterpret_cast<float *>(tab + kMaxTablePairs);
    float *nst = kt + kMaxTablePairs;
    float *c32 = nst + kMaxTablePairs;
    float *s32 = c32 + kMaxTablePairs;

    const int half = p.head_dim >> 1;
    const int n_table = p.num_slots * half;
    for (int i = threadIdx.x; i < n_table; i += kThreads) {
        const float2 cc = split16(p.cs[2 * i]), ss = split16(p.cs[2 * i + 1]);
        tab[i] = make_float4(cc.x, cc.y, ss.x, ss.y);
        c32[i] = __fadd_rn(cc.x, cc.y);   // fp32 cos (within one ulp of the fp64 value)
        s32[i] = __fadd_rn(ss.x, ss.y);
        kt[i] = bound_scale(c32[i], s32[i]);
        nst[i] = -s32[i];
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(&full[warp][s], 1);
        fence_mbar_init();
    }
    __syncthreads();

    const uint32_t first = blockIdx.x * kW + warp;
    const uint32_t stride = gridDim.x * kW;
    const uint32_t npairs = p.total_chunks / 2;
    const uint32_t n = npairs > first ? 2 * ((npairs - first + stride - 1) / stride) : 0;
    const int lane_v = lane & ((p.head_dim >> 4) - 1);
    uint8_t *wbuf = smem + (size_t)warp * kStages * kItemBytes;

    // Item j: pair j / 2 of the warp (pairs first, first + stride, ...), K if j is even, V if
    // odd. Lane 0 walks the pairs by additions and writes a pair's two Items at once, the V
    // Item into entry (j + 1) % kRing, whose previous item (j + 1 - kRing) has been read.
    if (lane == 0 && n > 0) {
        PairWalk w;
        w.pr = first;
        w.stride = stride;
        w.npairs = npairs;
        w.enter<kPaged>(p);
        walks[warp] = w;
    }
    const uint32_t row_bytes = (uint32_t)p.head_dim * 2;
    auto produce = [&](uint32_t j) {
        const uint32_t s = j % kStages;
        Item it;
        if ((j & 1u) == 0) {
            PairWalk w = walks[warp];
            if (j > 0) {
                w.next<kPaged>(p);
                walks[warp] = w;
            }
            const Pair q = pair_of<kPaged>(p, w);
            Item v = half_item(q, true);
            it = half_item(q, false);
            it.bytes = v.bytes = (uint32_t)q.rows * row_bytes;
            items[warp][j % kRing] = it;
            items[warp][(j + 1) % kRing] = v;
        } else {
            it = items[warp][j % kRing];
        }
        // bounds-checked builds: a source outside the slot's fragment is not copied (the
        // stage keeps stale bytes, the barrier completes without them)
        const bool src_ok = CM_IN_BOUNDS(it.src, it.bytes, it.src_base, it.src_size);
        mbar_arrive_expect_tx(&full[warp][s], src_ok ? it.bytes : 0u);
        if (j == 0 && p.withhold_warp == first + 1) return;   // injected: the wait runs out
        if (src_ok) bulk_load(wbuf + (size_t)s * kItemBytes, it.src, it.bytes, &full[warp][s]);
    };

    uint32_t produced = 0;
    if (lane == 0)
        for (; produced < n && produced < (uint32_t)kStages; ++produced) produce(produced);

    uint32_t i = 0;
    bool aborted = false;
    for (; i < n; ++i) {
        const uint32_t s = i % kStages;
        const bool ok = mbar_wait(&full[warp][s], (i / kStages) & 1u);
        if (__any_sync(0xFFFFFFFFu, !ok)) {
            aborted = true;
            break;
        }
        const Item it = items[warp][i % kRing];
        const uint8_t *buf = wbuf + (size_t)s * kItemBytes;
        if (it.rotate)
            rotate_from_smem<kPaged>(p, tab, kt, nst, c32, s32, it, buf, lane, lane_v);
        else
            copy_from_smem<kPaged>(p, it, buf, lane);
        __syncwarp();                          // every lane is done reading stage s
        if (lane == 0 && produced < n) {
            fence_proxy_async_smem();
            produce(produced++);               // item i + kStages into stage s
        }
    }
    if (aborted && lane == 0) {
        atomicOr(p.error, 1u);
        for (uint32_t j = i; j < produced; ++j)
            mbar_wait(&full[warp][j % kStages], (j / kStages) & 1u);
    }
}

template <bool kPaged, int kW, int kStages = kStagesDefault, int kMinBlocks = 16 / kW>
cudaError_t set_smem_attribute() {
    return cudaFuncSetAttribute(render_kernel<kPaged, kW, kStages, kMinBlocks>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)dyn_smem<kW, kStages>());
}

// ---------------------------------------------------------------- full-SM render

constexpr int kRegThreads = 256;           // 8 warps per CTA
constexpr int kRegBlocksPerSm = 3;         // 24 warps per SM
constexpr uint32_t kRegItemBytes = 1024;   // one work item: 2 vectors per lane
constexpr int kRegVecs = kRegItemBytes / 16 / 32;

// Paged outputs: where the rows of a pair go, for K and V alike (the two halves differ only
// in their pool). When the block size is a power of two no smaller than the pair's row
// count, the rows lie in at most two logical blocks: row r goes to half + da + r * stride
// before the block boundary (r < split), to half + db + r * stride after it, the block
// table read once per pair; otherwise (fast false) every row looks its block up.
struct PagedOffsets {
    int64_t da, db, stride;
    int split;
    bool fast;
};

__device__ __forceinline__ PagedOffsets paged_offsets(const RenderParams &p, int64_t pos0, int rows) {
    PagedOffsets o;
    o.fast = p.log2_block_size >= 0 && (int64_t)rows <= p.block_size;
    o.stride = p.stride_token * 2;
    o.split = rows;
    o.da = o.db = 0;
    if (o.fast) {
        const int64_t b0 = pos0 >> p.log2_block_size;
        const int64_t o0 = pos0 & (p.block_size - 1);
        const int64_t k = p.block_size - o0;                 // rows left in block b0
        o.da = table_entry(p, b0) * p.stride_block * 2 + o0 * o.stride;
        if (k < rows) {
            o.split = (int)k;
            o.db = table_entry(p, b0 + 1) * p.stride_block * 2 - k * o.stride;
        }
    }
    return o;
}

// Row r of one half of a pair (half = the half's item).
template <bool kPaged>
__device__ __forceinline__ uint4 *pair_row(const RenderParams &p, const Item &half,
                                           const PagedOffsets &po, int r) {
    if (!kPaged) return reinterpret_cast<uint4 *>(half.dst) + (int64_t)r * (p.head_dim >> 3);
    if (po.fast)
        return reinterpret_cast<uint4 *>(half.dst + (r < po.split ? po.da : po.db) + (int64_t)r * po.stride);
    PagedRows slow{};
    slow.fast = false;
    return row_dst<true>(p, half, r, slow);
}

// Stores vector v (0 <= v < rows * d / 8) of a copied item.
template <bool kPaged>
__device__ __forceinline__ void store_vec(const RenderParams &p, const Item &it,
                                          const PagedOffsets &po, int v, const uint4 &x) {
    const int log2_vpr = p.log2_pairs_per_row + 1;   // vectors per row = d / 8
    uint4 *d = pair_row<kPaged>(p, it, po, v >> log2_vpr) + (v & ((1 << log2_vpr) - 1));
    if (CM_IN_BOUNDS(d, 16, it.dst_base, it.dst_size)) st_stream(d, x);
}

// Full-SM render: persistent, kRegBlocksPerSm CTAs of 8 warps per SM, no shared-memory
// staging and no waits. Per pair, each lane loads its 2 vectors of the K item (for a
// rotated item: vector v of the first and of the second half of one row, v = lane mod
// (d/16)) and its 2 vectors of the V item, then stores V, then rotates (slots at a
// nonzero offset) and stores K. The lane's 8 (cos, sin) values are reloaded only when
// the slot changes.
template <bool kPaged>
__global__ void __launch_bounds__(kRegThreads, kRegBlocksPerSm)
render_reg_kernel(const __grid_constant__ RenderParams p) {
    __shared__ float4 tab[kMaxTablePairs];   // (c1, c2, s1, s2) for the second level
    __shared__ __align__(16) float kt[kMaxTablePairs];   // first-level bound scale per frequency
    __shared__ __align__(16) float nst[kMaxTablePairs];  // -s32 per frequency
    const int half = p.head_dim >> 1;
    const int n_table = p.num_slots * half;
    for (int i = threadIdx.x; i < n_table; i += kRegThreads) {
        const float2 cc = split16(p.cs[2 * i]), ss = split16(p.cs[2 * i + 1]);
        tab[i] = make_float4(cc.x, cc.y, ss.x, ss.y);
        kt[i] = bound_scale(__fadd_rn(cc.x, cc.y), __fadd_rn(ss.x, ss.y));
        nst[i] = -__fadd_rn(ss.x, ss.y);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    PairWalk w;
    w.pr = blockIdx.x * (kRegThreads / 32) + warp;
    w.stride = gridDim.x * (kRegThreads / 32);
    w.npairs = p.total_chunks / 2;
    if (w.pr >= w.npairs) return;
    w.enter<kPaged>(p);
    const int half_vecs = p.head_dim >> 4;
    const int vecs_per_row = p.head_dim >> 3;
    const int log2_hv = p.log2_pairs_per_row;
    const int lane_v = lane & (half_vecs - 1);
    int cur = -1;
    float c[8], s[8];
    do {
        const Pair q = pair_of<kPaged>(p, w);
        const int n_vec = q.rows * vecs_per_row;
        const int n_pairs = q.rows * half_vecs;
        const uint4 *ks = reinterpret_cast<const uint4 *>(q.ks);
        const uint4 *vs = reinterpret_cast<const uint4 *>(q.vs);
        uint4 rk[kRegVecs], rv[kRegVecs];
        if (q.rotate) {
#pragma unroll
            for (int k = 0; k < kRegVecs / 2; ++k) {
                const int qq = lane + 32 * k;
                const int off = (qq >> log2_hv) * vecs_per_row + lane_v;
                rk[2 * k] = rk[2 * k + 1] = make_uint4(0, 0, 0, 0);
                if (qq < n_pairs && CM_IN_BOUNDS(ks + off, 16, q.ks_base, q.src_size) &&
                    CM_IN_BOUNDS(ks + off + half_vecs, 16, q.ks_base, q.src_size)) {
                    rk[2 * k] = __ldcs(ks + off);
                    rk[2 * k + 1] = __ldcs(ks + off + half_vecs);
                }
            }
        } else {
#pragma unroll
            for (int u = 0; u < kRegVecs; ++u) {
                const int v = lane + 32 * u;
                rk[u] = make_uint4(0, 0, 0, 0);
                if (v < n_vec && CM_IN_BOUNDS(ks + v, 16, q.ks_base, q.src_size)) rk[u] = __ldcs(ks + v);
            }
        }
#pragma unroll
        for (int u = 0; u < kRegVecs; ++u) {
            const int v = lane + 32 * u;
            rv[u] = make_uint4(0, 0, 0, 0);
            if (v < n_vec && CM_IN_BOUNDS(vs + v, 16, q.vs_base, q.src_size)) rv[u] = __ldcs(vs + v);
        }
        PagedOffsets po{};
        if (kPaged) po = paged_offsets(p, q.pos0, q.rows);
        const Item vi = half_item(q, true);
#pragma unroll
        for (int u = 0; u < kRegVecs; ++u)
            if (lane + 32 * u < n_vec) store_vec<kPaged>(p, vi, po, lane + 32 * u, rv[u]);
        const Item ki = half_item(q, false);
        if (q.rotate) {
            if (q.cs_index != cur) {
                cur = q.cs_index;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float4 t = tab[cur + 8 * lane_v + e];
                    c[e] = __fadd_rn(t.x, t.y);   // (c32, s32) = (fl(c1 + c2), fl(s1 + s2))
                    s[e] = __fadd_rn(t.z, t.w);
                }
            }
#pragma unroll
            for (int k = 0; k < kRegVecs / 2; ++k) {
                const int qq = lane + 32 * k;
                if (qq < n_pairs) {
                    // copies of the two vectors, which the fix-up also reads
                    const uint4 a = rk[2 * k], b = rk[2 * k + 1];
                    const float4 ka = *reinterpret_cast<const float4 *>(kt + cur + 8 * lane_v);
                    const float4 kb = *reinterpret_cast<const float4 *>(kt + cur + 8 * lane_v + 4);
                    const float4 na = *reinterpret_cast<const float4 *>(nst + cur + 8 * lane_v);
                    const float4 nb = *reinterpret_cast<const float4 *>(nst + cur + 8 * lane_v + 4);
                    uint4 ao, bo;
                    uint32_t b0, b1, b2, b3;
                    rotate_word(a.x, b.x, c[0], s[0], na.x, ka.x, c[1], s[1], na.y, ka.y, ao.x, bo.x, b0);
                    rotate_word(a.y, b.y, c[2], s[2], na.z, ka.z, c[3], s[3], na.w, ka.w, ao.y, bo.y, b1);
                    rotate_word(a.z, b.z, c[4], s[4], nb.x, kb.x, c[5], s[5], nb.y, kb.y, ao.z, bo.z, b2);
                    rotate_word(a.w, b.w, c[6], s[6], nb.z, kb.z, c[7], s[7], nb.w, kb.w, ao.w, bo.w, b3);
                    if ((b0 | b1 | b2 | b3) != 0u)
                        fixup_pair(p, tab, cur + 8 * lane_v, a, b, b0, b1, b2, b3, ao, bo);
                    uint4 *d = pair_row<kPaged>(p, ki, po, qq >> log2_hv) + lane_v;
                    if (CM_IN_BOUNDS(d, 16, ki.dst_base, ki.dst_size)) st_stream(d, ao);
                    if (CM_IN_BOUNDS(d + half_vecs, 16, ki.dst_base, ki.dst_size))
                        st_stream(d + half_vecs, bo);
                }
            }
        } else {
#pragma unroll
            for (int u = 0; u < kRegVecs; ++u)
                if (lane + 32 * u < n_vec) store_vec<kPaged>(p, ki, po, lane + 32 * u, rk[u]);
        }
    } while (w.next<kPaged>(p));
}

}  // namespace

CM_DEFINE_BOUNDS_READER(take_render_bounds_violations)

cudaError_t render_prepare() {
    cudaError_t e = set_smem_attribute<false, 8>();
    if (e == cudaSuccess) e = set_smem_attribute<true, 8>();
    if (e == cudaSuccess) e = set_smem_attribute<false, 4, 6, 4>();
    if (e == cudaSuccess) e = set_smem_attribute<true, 4, 6, 4>();
    return e;
}

uint32_t render_item_bytes(RenderWidth w) {
    return (w == RenderWidth::kHalf || w == RenderWidth::kBeside) ? kItemBytes : kRegItemBytes;
}

int render_grid(uint64_t chunks, int num_sms, RenderWidth w) {
    if (w == RenderWidth::kHalf || w == RenderWidth::kBeside)
        return (int)std::max<uint64_t>(1, std::min<uint64_t>(chunks, (uint64_t)num_sms));
    const uint64_t ctas = (chunks / 2 + kRegThreads / 32 - 1) / (kRegThreads / 32);
    const uint64_t per_sm = w == RenderWidth::kFull ? (uint64_t)kRegBlocksPerSm : 1;
    return (int)std::max<uint64_t>(1, std::min<uint64_t>(ctas, per_sm * num_sms));
}

cudaError_t launch_render(const RenderParams &p, int grid, RenderWidth w, cudaStream_t stream) {
    if (p.total_chunks == 0) return cudaSuccess;
    switch (w) {
        case RenderWidth::kHalf:
            if (p.paged)
                render_kernel<true, 8><<<grid, 8 * 32, dyn_smem<8>(), stream>>>(p);
            else
                render_kernel<false, 8><<<grid, 8 * 32, dyn_smem<8>(), stream>>>(p);
            break;
        case RenderWidth::kBeside:
            if (p.paged)
                render_kernel<true, 4, 6, 4><<<grid, 4 * 32, dyn_smem<4, 6>(), stream>>>(p);
            else
                render_kernel<false, 4, 6, 4><<<grid, 4 * 32, dyn_smem<4, 6>(), stream>>>(p);
            break;
        default:   // kFull, kBesideSmall: the register kernel (grid sizes differ)
            if (p.paged)
                render_reg_kernel<true><<<grid, kRegThreads, 0, stream>>>(p);
            else
                render_reg_kernel<false><<<grid, kRegThreads, 0, stream>>>(p);
            break;
    }
    return cudaGetLastError();
}

}  // namespace cm
