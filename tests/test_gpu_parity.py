"""GPU parity: the CUDA library through its C ABI against the CPU oracle.

Bar: content addresses, norm keys, set membership, canonical order and V are
bit-exact; K is within 1 bf16 ulp per element (the non-exact count is also
asserted to be 0: the kernel certifies its fp32 rounding and recomputes the
rest in fp64 exactly as the oracle does). Every render is also byte-identical
across all delivery orders of its set.
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
from oracle.bf16 import is_nan_bits
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, gpu_fragments, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _render(ctx, deliveries, cap=None, fill=None):
    S = cm.FragmentSet(ctx)
    absorbed = [S.ingest(K, V)[1] for K, V in deliveries]
    K0 = deliveries[0][0]
    L, H, _, d = K0.shape
    total = S.seq_len()
    k_out, v_out = empty_out(L, H, cap or max(total, 1), d, fill=fill)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    S.close()
    return k_out, v_out, n, order, absorbed


# ---------------------------------------------------------------- content address + norm key

ID_SHAPES = [(4, 2, 37, 64), (4, 2, 53, 64), (1, 1, 1, 16), (2, 3, 1, 512), (3, 1, 5, 16),
             (2, 2, 33, 32), (5, 2, 7, 256), (28, 8, 9, 128), (1, 1, 300, 128),
             (3, 8, 70, 64), (2, 4, 129, 512)]


@pytest.mark.parametrize("shape", ID_SHAPES)
def test_fragment_id_and_norm_key_match_oracle(ctx, shape):
    L, H, T, d = shape
    g = torch.Generator(device="cuda:0").manual_seed(sum(shape))
    K = (torch.randn(shape, generator=g, device="cuda:0") * 1.3).to(torch.bfloat16)
    V = torch.randn(shape, generator=g, device="cuda:0").to(torch.bfloat16)
    fid, Q = ctx.fragment_id(K, V)
    ref = oracle_fragment(K, V)
    assert fid == ref.fid
    assert np.array_equal(np.array(Q, dtype=np.uint64), ref.Q)


def test_fragment_id_matches_the_frozen_golden_ids(ctx):
    # the ids recorded in tests/golden/content_address_ids.json by the oracle
    import importlib.util
    import json
    import os
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    spec = importlib.util.spec_from_file_location("_golden_ca", os.path.join(here, "content_address_ids.py"))
    gen = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(gen)
    with open(os.path.join(here, "content_address_ids.json")) as fh:
        rows = json.load(fh)["fragments"]
    for row in rows:
        Kb, Vb = gen.fragment_bits(row["shape"], row["seed"])
        K = torch.from_numpy(Kb.view(np.int16)).to("cuda:0").view(torch.bfloat16)
        V = torch.from_numpy(Vb.view(np.int16)).to("cuda:0").view(torch.bfloat16)
        fid, _ = ctx.fragment_id(K, V)
        assert fid.hex() == row["id_hex"], row["name"]


def test_norm_key_special_values(ctx):
    L, H, T, d = 2, 2, 6, 16
    K = torch.zeros((L, H, T, d), dtype=torch.bfloat16, device="cuda:0")
    V = torch.zeros_like(K)
    Kb = K.view(torch.int16)
    Kb[1, 0, 0, :] = 0x7F7F           # largest finite: saturates
    Kb[1, 0, 1, 3] = 0x7FC0           # NaN: saturates
    Kb[1, 1, 2, 5] = -0x8000 + 0x0001  # negative subnormal (0x8001)
    Kb[1, 1, 3, :] = 0x3F80           # ones: norm 4
    fid, Q = ctx.fragment_id(K, V)
    ref = oracle_fragment(K, V)
    assert fid == ref.fid
    assert np.array_equal(np.array(Q, dtype=np.uint64), ref.Q)


def test_norm_key_rounds_exact_halves_to_even(ctx):
    # rows of 16 equal entries k 2^-23: 2^20 n = k / 2 exactly, rounded half to even
    # (0, 2, 2, 4, 4 for k = 1, 3, 5, 7, 9), for one head and summed over two
    ks, want = [1, 3, 5, 7, 9], [0, 2, 2, 4, 4]
    for H in (1, 2):
        K = torch.zeros((2, H, len(ks), 16), dtype=torch.bfloat16, device="cuda:0")
        for t, k in enumerate(ks):
            K[1, :, t, :] = k * 2.0 ** -23
        V = torch.zeros_like(K)
        fid, Q = ctx.fragment_id(K, V)
        assert list(Q) == [H * q for q in want]
        ref = oracle_fragment(K, V)
        assert fid == ref.fid and np.array_equal(np.array(Q, dtype=np.uint64), ref.Q)


def test_norm_key_wide_exponent_range(ctx):
    # routing-layer rows whose elements span up to 2^40 in magnitude (most fp64 row sums
    # round; rows with large elements saturate), with zeros, subnormals and infinities
    # mixed into some vectors: every exponent field of the bf16 -> fp64 conversion, and
    # both the integer conversion of all-normal vectors and the fp32 one of the others
    L, H, T, d = 3, 4, 150, 64                      # 600 rows of K[1]: several norm blocks
    rng = np.random.default_rng(2607)
    bits = rng.integers(0, 1 << 16, size=(L, H, T, d), dtype=np.uint32).astype(np.uint16)
    rows = bits[1].reshape(H * T, d)
    emax = rng.integers(115, 161, size=(H * T, 1))   # largest element 2^-12 .. 2^33
    expo = np.clip(emax - rng.integers(0, 41, size=(H * T, d)), 1, 254)
    sign = rng.integers(0, 2, size=(H * T, d)) << 15
    rows[:] = (sign | (expo << 7) | rng.integers(0, 128, size=(H * T, d))).astype(np.uint16)
    odd = rng.random((H * T, d)) < 0.03
    rows[odd] = (rng.integers(0, 2, size=int(odd.sum())) << 15 |
                 rng.integers(0, 128, size=int(odd.sum()))).astype(np.uint16)   # zeros, subnormals
    rows[7, 3] = 0x7F80                             # +inf
    rows[400, 60] = 0xFF80                          # -inf
    rows[9, :] = rng.integers(1, 128, size=d).astype(np.uint16)   # all subnormal
    K = torch.from_numpy(bits.view(np.int16)).to("cuda:0").view(torch.bfloat16)
    V = torch.zeros_like(K)
    fid, Q = ctx.fragment_id(K, V)
    ref = oracle_fragment(K, V)
    assert fid == ref.fid
    got = np.array(Q, dtype=np.uint64)
    assert np.array_equal(got, ref.Q)
    sat = np.uint64((1 << 44) - 1)
    assert (got >= sat).any() and (got < sat).any()   # positions with and without a saturated head


# ---------------------------------------------------------------- tiny workload: every order

def test_tiny_all_delivery_orders_match_oracle(ctx):
    w, frags, sched = gpu_fragments("tiny")
    msgs = [(frags[i][0].clone(), frags[i][1].clone()) for i in sched]
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    first = None
    for perm in itertools.permutations(range(len(msgs))):
        k_out, v_out, n, order, absorbed = _render(ctx, [msgs[i] for i in perm])
        assert sum(absorbed) == 1 and n == K_ref.shape[2] == 37 + 53
        assert order == [f.fid for f in o_order]
        kb, vb = synthetic.to_bits(k_out), synthetic.to_bits(v_out)
        assert np.array_equal(vb, V_ref)
        assert assert_k_parity(kb, K_ref) == 0
        if first is None:
            first = (kb, vb)
        assert np.array_equal(kb, first[0]) and np.array_equal(vb, first[1])


# ---------------------------------------------------------------- Qwen3-1.7B shaped, N = 2

def test_q17_n2_full_parity(ctx):
    w, frags, sched = gpu_fragments("q17_n2")
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    results = []
    for perm in itertools.permutations(range(2)):
        k_out, v_out, n, order, absorbed = _render(ctx, [frags[i] for i in perm])
        assert n == 1024 and order == [f.fid for f in o_order] and not any(absorbed)
        results.append((synthetic.to_bits(k_out), synthetic.to_bits(v_out)))
    kb, vb = results[0]
    assert np.array_equal(vb, V_ref)
    assert assert_k_parity(kb, K_ref) == 0
    assert np.array_equal(results[1][0], kb) and np.array_equal(results[1][1], vb)


# ---------------------------------------------------------------- rounding edge cases

def test_rotation_of_special_values_matches_oracle(ctx):
    L, H, T, d = 1, 2, 64, 128
    rng = np.random.default_rng(3)
    bits = rng.integers(0, 1 << 16, size=(L, H, T, d), dtype=np.uint64).astype(np.uint16)
    # avoid NaN payload patterns, keep +-inf, +-0, subnormals, the largest finites
    nan = ((bits & 0x7F80) == 0x7F80) & ((bits & 0x7F) != 0)
    bits[nan] = 0x3F80
    bits[0, 0, 0, :8] = [0x0000, 0x8000, 0x0001, 0x8001, 0x007F, 0x7F7F, 0xFF7F, 0x7F80]
    bits[0, 0, 0, 64:72] = [0x8000, 0x0000, 0x0001, 0x0002, 0x807F, 0x7F7F, 0x7F7F, 0x3F80]
    bits[0, 1, :, :] = (bits[0, 1, :, :] & 0x80FF) | 0x0000   # many subnormals
    base = torch.from_numpy(bits.view(np.int16)).to("cuda:0").view(torch.bfloat16)
    lead = torch.zeros((L, H, 1000, d), dtype=torch.bfloat16, device="cuda:0")
    frags = [(lead, lead.clone()), (base.contiguous(), base.clone())]
    k_out, v_out = empty_out(L, H, 1000 + T, d)
    n = ctx.bagmerge(frags, k_out, v_out)
    torch.cuda.synchronize()
    assert n == 1000 + T
    ref = oracle.rotate_k(bits, 1000, THETA)
    got = synthetic.to_bits(k_out)[:, :, 1000:]
    assert assert_k_parity(got, ref) == 0


# numpy warns when it widens a signalling NaN payload; the oracle's result is still NaN
@pytest.mark.filterwarnings("ignore:invalid value encountered in cast:RuntimeWarning")
def test_nan_and_inf_inputs_hash_as_bytes_and_propagate():
    # NaN and inf are bytes to the content address and IEEE values to the rotation: ids
    # equal the oracle's, V and the first slot's K (byte copies) keep every NaN payload,
    # and the rotated K is NaN exactly where the oracle's is (within 1 ulp elsewhere). The
    # routing layer 1 holds no NaN, so the norm keys stay finite and order the two.
    L, H, d = 3, 2, 64
    rng = np.random.default_rng(21)
    specials = np.array([0x7FC1, 0xFFA0, 0x7F81, 0xFFFF, 0x7F80, 0xFF80], dtype=np.uint16)
    frags, bits = [], []
    for T, sc in ((20, 2.0), (33, 0.5)):
        K = (rng.standard_normal((L, H, T, d)) * sc).astype(np.float32)
        V = rng.standard_normal((L, H, T, d)).astype(np.float32)
        kb = (K.view(np.uint32) >> 16).astype(np.uint16)
        vb = (V.view(np.uint32) >> 16).astype(np.uint16)
        for arr in (kb, vb):
            for layer in (0, 2):
                idx = rng.integers(0, arr[layer].size, size=12)
                arr[layer].reshape(-1)[idx] = rng.choice(specials, size=12)
        bits.append((kb, vb))
        frags.append(tuple(torch.from_numpy(a.view(np.int16)).to("cuda:0").view(torch.bfloat16)
                           for a in (kb, vb)))
    refs = [oracle.make_fragment(kb, vb) for kb, vb in bits]
    c = cm.Context(0, THETA)
    S = cm.FragmentSet(c)
    res = S.ingest_batch(frags)
    assert [r[0] for r in res] == [f.fid for f in refs]
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(refs), THETA)
    assert order == [f.fid for f in o_order] and order[0] == refs[0].fid
    kg, vg = synthetic.to_bits(k_out), synthetic.to_bits(v_out)
    assert np.array_equal(vg, V_ref) and np.array_equal(vg[:, :, :20], bits[0][1])
    assert np.array_equal(kg[:, :, :20], bits[0][0])        # slot 0: bytes, payloads kept
    assert is_nan_bits(kg[:, :, 20:]).any()
    assert assert_k_parity(kg, K_ref) == 0
    S.close()
    c.close()


# ---------------------------------------------------------------- layout, capacity, canaries

@pytest.mark.parametrize("d", [16, 64, 256, 512])
def test_render_layout_with_capacity_and_canaries(ctx, d):
    L, H = 3, 2
    lengths = [1, 129, 70, 600]
    g = torch.Generator(device="cuda:0").manual_seed(d)
    frags = []
    for i, T in enumerate(lengths):
        K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.6 + 0.3 * i)).to(torch.bfloat16)
        V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
        frags.append((K, V))
    total = sum(lengths)
    cap = total + 37
    k_out, v_out, n, order, _ = _render(ctx, frags, cap=cap, fill=0x5A5A)
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    assert n == total and order == [f.fid for f in o_order]
    kb, vb = synthetic.to_bits(k_out), synthetic.to_bits(v_out)
    assert np.array_equal(vb[:, :, :total], V_ref)
    assert assert_k_parity(kb[:, :, :total], K_ref) == 0
    assert (kb[:, :, total:] == 0x5A5A).all() and (vb[:, :, total:] == 0x5A5A).all()


def test_bagmerge_explicit_order_and_naive_redelivery(ctx):
    w, frags, _ = gpu_fragments("tiny")
    a, b = frags
    ref = [oracle_fragment(K, V) for K, V in frags]
    for order_idx in ([0, 1], [1, 0], [0, 1, 0, 1, 0, 1]):
        seq = [frags[i] for i in order_idx]
        L, H, _, d = a[0].shape
        total = sum(f[0].shape[2] for f in seq)
        k_out, v_out = empty_out(L, H, total, d)
        n = ctx.bagmerge(seq, k_out, v_out)
        torch.cuda.synchronize()
        K_ref, V_ref = oracle.bagmerge([ref[i] for i in order_idx], THETA)
        assert n == total
        assert np.array_equal(synthetic.to_bits(v_out), V_ref)
        assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0


def test_empty_set_renders_nothing(ctx):
    S = cm.FragmentSet(ctx)
    n, order = cm.cm_render(S.handle, 0, 0, 0)
    assert n == 0 and order == []
    S.close()


# ---------------------------------------------------------------- ABI errors on the GPU path

def test_abi_errors(ctx):
    g = torch.Generator(device="cuda:0").manual_seed(1)
    K = torch.randn((2, 2, 8, 64), generator=g, device="cuda:0").to(torch.bfloat16)
    V = torch.randn((2, 2, 8, 64), generator=g, device="cuda:0").to(torch.bfloat16)
    S = cm.FragmentSet(ctx)
    S.ingest(K, V)
    K2 = torch.zeros((2, 2, 8, 32), dtype=torch.bfloat16, device="cuda:0")
    with pytest.raises(cm.CMError) as e:
        S.ingest(K2, K2.clone())
    assert e.value.status == cm.Status.ERR_SHAPE_MISMATCH
    # odd head_dim / not a power of two
    bad = cm.cm_fragment(2, 2, 8, 48, K.data_ptr(), V.data_ptr())
    with pytest.raises(cm.CMError) as e:
        cm.cm_ingest(S.handle, bad)
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    # misaligned pointer
    mis = cm.cm_fragment(2, 2, 8, 64, K.data_ptr() + 2, V.data_ptr())
    with pytest.raises(cm.CMError) as e:
        cm.cm_ingest(S.handle, mis)
    assert e.value.status == cm.Status.ERR_ALIGNMENT
    # capacity too small
    k_out, v_out = empty_out(2, 2, 7, 64)
    with pytest.raises(cm.CMError) as e:
        S.render(k_out, v_out)
    assert e.value.status == cm.Status.ERR_CAPACITY
    # union across contexts
    other = cm.Context(0, THETA)
    S2 = cm.FragmentSet(other)
    with pytest.raises(cm.CMError) as e:
        S.union(S2)
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    S2.close()
    other.close()
    # routing layer out of range
    c3 = cm.Context(0, THETA, routing_layer=5)
    with pytest.raises(cm.CMError) as e:
        c3.fragment_id(K, V)
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    c3.close()
    S.close()


def test_verify_bytes_on_hit_accepts_true_duplicates(ctx):
    c = cm.Context(0, THETA, verify_bytes_on_hit=True)
    g = torch.Generator(device="cuda:0").manual_seed(2)
    K = torch.randn((2, 2, 9, 64), generator=g, device="cuda:0").to(torch.bfloat16)
    V = torch.randn((2, 2, 9, 64), generator=g, device="cuda:0").to(torch.bfloat16)
    S = cm.FragmentSet(c)
    assert S.ingest(K, V)[1] is False
    assert S.ingest(K.clone(), V.clone())[1] is True
    assert len(S) == 1
    S.close()
    c.close()


def test_verify_bytes_on_hit_reports_a_collision(ctx):
    # an id hit whose bytes differ, made by breaking the borrow contract on purpose: the
    # set's record is changed in place after its ingest, then the original bytes arrive
    # again and hash to the stored id
    c = cm.Context(0, THETA, verify_bytes_on_hit=True)
    g = torch.Generator(device="cuda:0").manual_seed(3)
    mk = lambda T: (torch.randn((2, 2, T, 64), generator=g, device="cuda:0").to(torch.bfloat16),
                    torch.randn((2, 2, T, 64), generator=g, device="cuda:0").to(torch.bfloat16))
    (K, V), B, C = mk(9), mk(5), mk(7)
    K0, V0 = K.clone(), V.clone()
    S = cm.FragmentSet(c)
    fid, _ = S.ingest(K, V)
    V.view(torch.int16)[1, 1, 8, 63] ^= 1
    with pytest.raises(cm.CMError) as e:
        S.ingest(K0, V0)
    assert e.value.status == cm.Status.ERR_COLLISION
    assert len(S) == 1
    # in a batch the deliveries before the colliding one are inserted, the later ones
    # are not processed (as n single calls that stop at the failing one)
    with pytest.raises(cm.CMError) as e:
        S.ingest_batch([B, (K0, V0), C])
    assert e.value.status == cm.Status.ERR_COLLISION
    assert len(S) == 2 and S.ids() == sorted([fid, oracle_fragment(*B).fid])
    assert any(kv[0] is B[0] for kv in S._held)     # the binding keeps B's tensors alive
    # with the record's bytes restored the same delivery is absorbed again
    V.copy_(V0)
    assert S.ingest(K0, V0) == (fid, True)
    # without verification an id hit is absorbed on the id alone
    c2 = cm.Context(0, THETA)
    S2 = cm.FragmentSet(c2)
    S2.ingest(K, V)
    V.view(torch.int16)[1, 1, 8, 63] ^= 1
    assert S2.ingest(K0, V0) == (fid, True)
    S2.close()
    c2.close()
    S.close()
    c.close()


# ---------------------------------------------------------------- union on the GPU-built sets

def test_union_algebra_and_render_invariance(ctx):
    w, frags, _ = gpu_fragments("q17_arity")
    frags = [(K[:, :, :64].contiguous(), V[:, :, :64].contiguous()) for K, V in frags]
    singles = []
    for K, V in frags:
        S = cm.FragmentSet(ctx)
        S.ingest(K, V)
        singles.append(S)
    L, H, _, d = frags[0][0].shape
    k0, v0 = empty_out(L, H, 64 * 5, d)
    ref_bits = None
    for perm in itertools.permutations(range(5)):
        U = cm.FragmentSet(ctx)
        for i in perm:
            U.union(singles[i])
        U.union(singles[perm[0]])          # idempotent / absorbing
        assert len(U) == 5
        n, order = U.render(k0, v0)
        torch.cuda.synchronize()
        kb = (synthetic.to_bits(k0), synthetic.to_bits(v0))
        if ref_bits is None:
            ref_bits = kb
        assert np.array_equal(kb[0], ref_bits[0]) and np.array_equal(kb[1], ref_bits[1])
        U.close()
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, _ = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    assert np.array_equal(ref_bits[1], V_ref)
    assert assert_k_parity(ref_bits[0], K_ref) == 0
    for S in singles:
        S.close()


# ---------------------------------------------------------------- launch-group boundaries

def test_roots_at_level_one_and_two(ctx):
    # 64 T bytes per fragment: T <= 256 gives at most 16 leaves, so level 1 is the root;
    # T = 257 has 17 leaves and its root at level 2 (one tree-top kernel per call: few
    # level-1 nodes)
    L, H, d = 1, 1, 16
    g = torch.Generator(device="cuda:0").manual_seed(16)
    frags = [(torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
             for T in (1, 15, 16, 17, 255, 256)]
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(frags)
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    assert t["inner_hash_launches"] == 1
    assert [r[0] for r in res] == [oracle_fragment(K, V).fid for K, V in frags]
    K, V = (torch.randn((L, H, 257, d), generator=g, device="cuda:0").to(torch.bfloat16)
            for _ in range(2))
    cm.cm_context_set_timing(ctx.handle, True)
    fid, _ = S.ingest(K, V)
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    assert t["inner_hash_launches"] == 1 and fid == oracle_fragment(K, V).fid
    S.close()


def test_forty_fragments_span_two_render_and_two_tree_top_calls(ctx):
    # more fragments than one render launch (32 slots) or one tree-top launch (32) holds
    L, H, d = 2, 1, 64
    g = torch.Generator(device="cuda:0").manual_seed(40)
    frags = []
    for i in range(40):
        T = 1 + (i * 37) % 50
        K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.5 + 0.02 * i)).to(torch.bfloat16)
        V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
        frags.append((K, V))
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(frags)
    total = S.seq_len()
    k_out, v_out = empty_out(L, H, total, d)
    n, order = S.render(k_out, v_out)
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    # two tree-top calls (32 + 8 fragments), one kernel each (few level-1 nodes)
    assert t["render_launches"] == 2 and t["inner_hash_launches"] == 2
    assert t["leaf_hash_launches"] == 2 and t["leaf_hash_fragments"] == 40
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    assert [r[0] for r in res] == [f.fid for f in ref_frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()


def test_head_dim_512_spans_table_limited_render_groups(ctx):
    # 1792 (cos, sin) pairs per launch = 7 slots at d = 512: nine fragments need two launches
    L, H, d = 2, 1, 512
    g = torch.Generator(device="cuda:0").manual_seed(512)
    frags = []
    for i in range(9):
        T = 3 + 5 * i
        K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.5 + 0.1 * i)).to(torch.bfloat16)
        V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
        frags.append((K, V))
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()


def test_long_fragment_and_large_offsets(ctx):
    # T = 40000 tokens in slot 0 pushes the other slots' offsets past 40000 (angles of
    # thousands of radians at the highest frequency)
    L, H, d = 1, 2, 128
    g = torch.Generator(device="cuda:0").manual_seed(9)
    big = ((torch.randn((L, H, 40000, d), generator=g, device="cuda:0") * 3).to(torch.bfloat16),
           torch.randn((L, H, 40000, d), generator=g, device="cuda:0").to(torch.bfloat16))
    small = [((torch.randn((L, H, T, d), generator=g, device="cuda:0") * 0.3).to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)) for T in (333, 4096)]
    frags = [big] + small
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    ref_frags = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(ref_frags), THETA)
    assert order == [f.fid for f in o_order] and order[0] == ref_frags[0].fid
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()


@pytest.mark.parametrize("L,H,d,lengths", [
    (1, 1, 16, (262145, 3, 1000)),      # 2^18 + 1 tokens: offsets past 262,144, 16,385 leaves
    (1, 64, 512, (37, 5)),              # many heads, 1 KiB rows (4 rows per work item)
    (80, 1, 16, (9, 70)),               # many layers (routing layer 40)
    (3, 8, 128, (1, 1, 1)),             # single-token fragments only (T* = 1)
])
def test_shape_extremes_match_oracle(ctx, L, H, d, lengths):
    g = torch.Generator(device="cuda:0").manual_seed(L * 1000 + H * 10 + d)
    # decreasing K scales: the first (longest) fragment leads the canonical order, so the
    # others are rotated by offsets of its length
    frags = [((torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.5 + len(lengths) - i))
              .to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
             for i, T in enumerate(lengths)]
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(frags)
    refs = [oracle_fragment(K, V) for K, V in frags]
    assert [r[0] for r in res] == [f.fid for f in refs]
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(refs), THETA)
    assert n == sum(lengths) and order == [f.fid for f in o_order] and order[0] == refs[0].fid
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()


@pytest.mark.parametrize("rl", [-1, 0, 2, 5])
def test_explicit_routing_layer(rl):
    # the routing layer l* picks whose norms order the set (Eq. rho); A's keys are large in
    # layers 0-2, B's in layers 3-5, C's in none, so A leads for l* < 3 and B for l* >= 3
    # (the default floor(6 / 2) = 3 included)
    L, H, d = 6, 2, 64
    c = cm.Context(0, THETA, routing_layer=rl)
    g = torch.Generator(device="cuda:0").manual_seed(50 + rl)
    lo = torch.tensor([3.0, 3.0, 3.0, 0.5, 0.5, 0.5], device="cuda:0").view(L, 1, 1, 1)
    scales = (lo, lo.flip(0), torch.ones_like(lo))
    frags = [((torch.randn((L, H, T, d), generator=g, device="cuda:0") * sc).to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
             for sc, T in zip(scales, (40, 27, 61))]
    refs = [oracle_fragment(K, V, routing_layer=rl) for K, V in frags]
    for (K, V), ref in zip(frags, refs):
        fid, q = c.fragment_id(K, V)
        assert fid == ref.fid and np.array_equal(np.array(q, dtype=np.uint64), ref.Q)
    S = cm.FragmentSet(c)
    S.ingest_batch(frags[::-1])
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    n, order = S.render(k_out, v_out)
    torch.cuda.synchronize()
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(refs), THETA)
    assert order == [f.fid for f in o_order]
    assert order[0] == refs[0 if 0 <= rl < 3 else 1].fid
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()
    c.close()


def test_exact_ties_order_by_id():
    # A, B and C tie exactly on S (Eq. rho over the last T* = 20 rows of K[l*]): A and B
    # share K and differ in V, C is 10 rows longer with the same last 20 rows at l*. D has
    # larger keys. Expected: D, then the tied three by descending id (big-endian), under
    # every delivery order, as the oracle orders them.
    L, H, d, rl = 4, 2, 64, 2
    g = torch.Generator(device="cuda:0").manual_seed(77)
    rnd = lambda T, sc=1.0: (torch.randn((L, H, T, d), generator=g, device="cuda:0") * sc).to(torch.bfloat16)
    K0 = rnd(20)
    A = (K0, rnd(20))
    B = (K0.clone(), rnd(20))
    KC = rnd(30)
    KC[rl, :, 10:] = K0[rl]
    C = (KC, rnd(30))
    D = (rnd(25, 4.0), rnd(25))
    frags = [A, B, C, D]
    refs = [oracle_fragment(K, V) for K, V in frags]
    assert len({f.fid for f in refs}) == 4
    tail = [int(f.Q[-20:].astype(object).sum()) for f in refs]
    assert tail[0] == tail[1] == tail[2] < tail[3]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(refs), THETA)
    want = [refs[3].fid] + sorted((f.fid for f in refs[:3]), reverse=True)
    assert [f.fid for f in o_order] == want
    c = cm.Context(0, THETA)
    for perm in itertools.permutations(range(4)):
        S = cm.FragmentSet(c)
        S.ingest_batch([frags[i] for i in perm])
        k_out, v_out = empty_out(L, H, S.seq_len(), d)
        n, order = S.render(k_out, v_out)
        torch.cuda.synchronize()
        assert order == want
        assert np.array_equal(synthetic.to_bits(v_out), V_ref)
        assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
        S.close()
    c.close()


def test_rendered_cache_as_a_fragment_is_the_foil(ctx):
    # Section 4.4's foil: a rendered cache M = render({A, B}) delivered again as a fragment
    # is a new element; render({M, B}) differs from render({A, B}). The GPU's M hashes to
    # the oracle's id of the oracle's M, and the second merge equals the oracle's.
    L, H, d = 3, 2, 64
    g = torch.Generator(device="cuda:0").manual_seed(88)
    rnd = lambda T, sc: (torch.randn((L, H, T, d), generator=g, device="cuda:0") * sc).to(torch.bfloat16)
    A, B = (rnd(23, 2.0), rnd(23, 1.0)), (rnd(17, 0.7), rnd(17, 1.0))
    S = cm.FragmentSet(ctx)
    S.ingest_batch([A, B])
    Mk, Mv = empty_out(L, H, 40, d)
    S.render(Mk, Mv)
    torch.cuda.synchronize()
    refs = [oracle_fragment(K, V) for K, V in (A, B)]
    K1, V1, _ = oracle.render(oracle.from_deliveries(refs), THETA)
    m_ref = oracle.make_fragment(K1, V1)
    T2 = cm.FragmentSet(ctx)
    res = T2.ingest_batch([(Mk, Mv), B])
    assert res[0] == (m_ref.fid, False) and res[0][0] not in S.ids()
    k2, v2 = empty_out(L, H, 57, d)
    n, order = T2.render(k2, v2)
    torch.cuda.synchronize()
    K2, V2, o2 = oracle.render(oracle.from_deliveries([m_ref, refs[1]]), THETA)
    assert n == 57 and order == [f.fid for f in o2]
    assert np.array_equal(synthetic.to_bits(v2), V2)
    assert assert_k_parity(synthetic.to_bits(k2), K2) == 0
    assert K2.shape != K1.shape
    S.close()
    T2.close()


# ---------------------------------------------------------------- rotation stress

@pytest.mark.parametrize("theta", [1.0e4, 1.0e6, 5.0e5, 1.0e40])
def test_rotation_stress_random_bit_patterns(theta):
    # every finite bf16 bit pattern is a possible key; many slots give many (cos, sin)
    # pairs, including tiny sines when theta is huge
    c = cm.Context(0, theta)
    L, H, d = 1, 2, 128
    rng = np.random.default_rng(int(theta) % 1000 + 1)
    frags, bits_list = [], []
    for i in range(12):
        T = int(rng.integers(1, 90))
        bits = rng.integers(0, 1 << 16, size=(L, H, T, d), dtype=np.uint64).astype(np.uint16)
        bits[((bits & 0x7F80) == 0x7F80)] &= 0xBF7F          # no inf / NaN
        K = torch.from_numpy(bits.view(np.int16)).to("cuda:0").view(torch.bfloat16)
        V = torch.from_numpy(rng.integers(0, 1 << 15, size=bits.shape).astype(np.int16)).to(
            "cuda:0").view(torch.bfloat16)
        frags.append((K.contiguous(), V.contiguous()))
        bits_list.append(bits)
    total = sum(f[0].shape[2] for f in frags)
    k_out, v_out = empty_out(L, H, total, d)
    n = c.bagmerge(frags, k_out, v_out)
    torch.cuda.synchronize()
    kb = synthetic.to_bits(k_out)
    s = 0
    for bits in bits_list:
        T = bits.shape[2]
        want = oracle.rotate_k(bits, s, theta)
        assert assert_k_parity(kb[:, :, s:s + T], want, f"slot@{s}") == 0
        s += T
    c.close()


def _midpoint_distance_ulps(z):
    """Distance of fp64 values z (normal range) to the nearest bf16 rounding midpoint, in
    fp32 ulps of z."""
    _, e = np.frexp(z)                          # z = m 2^e, 0.5 <= |m| < 1
    q = np.ldexp(1.0, e - 8)                    # the bf16 quantum of that binade
    m = (np.floor(z / q) + 0.5) * q
    return np.abs(z - m) / np.ldexp(1.0, e - 24)


@pytest.mark.parametrize("theta", [1.0e4, 1.0e6])
def test_rotation_near_rounding_midpoints(theta):
    # keys chosen so that their rotated values lie within a few fp32 ulps of a bf16
    # rounding midpoint, where the fp32 first level cannot certify them: the second level
    # and the fp64 level decide; the render must still equal the oracle bit for bit
    from oracle.bf16 import bits_to_f64
    from oracle.merge import delta_cos_sin
    c = cm.Context(0, theta)
    L, H, d, T = 1, 2, 128, 16
    half = d // 2
    rng = np.random.default_rng(int(theta) % 997)

    def rand_bf16(n):
        e = rng.integers(118, 134, size=n)
        return ((rng.integers(0, 2, size=n) << 15) | (e << 7) | rng.integers(0, 128, size=n)).astype(np.uint16)

    frags, bits_list, near = [], [], []
    for p, s in enumerate([0, T, 2 * T, 3 * T]):
        bits = np.empty((L, H, T, d), dtype=np.uint16)
        cs, sn = delta_cos_sin(s, d, theta)
        for j in range(half):
            # the H T pairs (x, y) of frequency j closest to a midpoint, out of 512 x 512
            xs, ys = rand_bf16(512), rand_bf16(512)
            if s == 0:
                ix, iy = rng.integers(0, 512, size=H * T), rng.integers(0, 512, size=H * T)
            else:
                x, y = bits_to_f64(xs)[:, None], bits_to_f64(ys)[None, :]
                dist = np.minimum(_midpoint_distance_ulps(x * cs[j] - y * sn[j]),
                                  _midpoint_distance_ulps(y * cs[j] + x * sn[j]))
                best = np.argsort(dist, axis=None)[:H * T]
                ix, iy = np.unravel_index(best, dist.shape)
                near.append(np.median(dist.ravel()[best]))
            bits[0, :, :, j] = xs[ix].reshape(H, T)
            bits[0, :, :, j + half] = ys[iy].reshape(H, T)
        K = torch.from_numpy(bits.view(np.int16)).to("cuda:0").view(torch.bfloat16).contiguous()
        V = torch.from_numpy(rng.integers(0, 1 << 15, size=bits.shape).astype(np.int16)).to(
            "cuda:0").view(torch.bfloat16).contiguous()
        frags.append((K, V))
        bits_list.append(bits)
    assert np.median(near) < 4.0          # the construction does land near the midpoints
    total = 4 * T
    k_out, v_out = empty_out(L, H, total, d)
    assert c.bagmerge(frags, k_out, v_out) == total
    torch.cuda.synchronize()
    kb = synthetic.to_bits(k_out)
    for p, bits in enumerate(bits_list):
        s = p * T
        want = oracle.rotate_k(bits, s, theta)
        assert assert_k_parity(kb[:, :, s:s + T], want, f"slot@{s}") == 0
    c.close()


# ---------------------------------------------------------------- concurrent use of one context

def test_two_threads_share_a_context(ctx):
    import threading
    results, errors = {}, []

    def worker(name, seed):
        try:
            stream = torch.cuda.Stream()
            with torch.cuda.stream(stream):
                frags = [((torch.randn((3, 2, T, 64), device="cuda:0") * (0.5 + 0.2 * i)).to(torch.bfloat16),
                          torch.randn((3, 2, T, 64), device="cuda:0").to(torch.bfloat16))
                         for i, T in enumerate([40 + seed, 77, 12 + seed])]
                outs = []
                for rep in range(5):
                    S = cm.FragmentSet(ctx)
                    S.ingest_batch(frags, stream)
                    k, v = empty_out(3, 2, S.seq_len(), 64)
                    S.render(k, v, stream)
                    stream.synchronize()
                    outs.append((synthetic.to_bits(k), synthetic.to_bits(v), S.ids()))
                    S.close()
            results[name] = (frags, outs)
        except Exception as e:     # surfaced below
            errors.append(e)

    threads = [threading.Thread(target=worker, args=(f"t{i}", i)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for name, (frags, outs) in results.items():
        ref = oracle.from_deliveries([oracle_fragment(K, V) for K, V in frags])
        K_ref, V_ref, _ = oracle.render(ref, THETA)
        for kb, vb, ids in outs:
            assert ids == ref.ids()
            assert np.array_equal(vb, V_ref)
            assert assert_k_parity(kb, K_ref) == 0


# ---------------------------------------------------------------- resources

def test_contexts_release_device_memory():
    # contexts created, used (scratch grown by a batch, timing events, the re-delivery fast
    # path, a render) and destroyed 20 times: the device's free memory returns to where it
    # was after the first cycle (every tensor here is allocated before the baseline)
    L, H, d = 4, 4, 128
    g = torch.Generator(device="cuda:0").manual_seed(99)
    frags = [((torch.randn((L, H, T, d), generator=g, device="cuda:0")).to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
             for T in (3000, 1700, 900)]
    copy = (frags[0][0].clone(), frags[0][1].clone())
    k, v = empty_out(L, H, 5600, d)

    def cycle():
        c = cm.Context(0, THETA)
        cm.cm_context_set_timing(c.handle, True)
        cm.cm_context_set_dedup_by_bytes(c.handle, True)
        S = cm.FragmentSet(c)
        S.ingest_batch(frags + [copy])
        n, _ = S.render(k, v)
        cm.cm_context_kernel_times(c.handle, reset=True)
        S.close()
        c.close()
        return n

    assert cycle() == 5600
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(20):
        cycle()
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    assert free0 - free1 < (4 << 20), (free0, free1)
