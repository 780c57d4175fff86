"""GPU parity at the benchmark's full sizes, in the launch configuration bench.py
times (one cm_ingest_render call: two replicas take half the fragments each, union,
render, with the render beside the content address), and at the full sizes of the
other workloads.

The oracle computes every content address and norm key in full (hashlib over all
bytes) and renders every (slot, layer, head) plane: V planes are compared bit for
bit, K planes within 1 bf16 ulp with the non-exact count asserted to be 0.
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
import synthetic
from oracle.content_address import fragment_id, id_as_int
from oracle.norm import norm_key, tail_sum
from parity_util import THETA, assert_k_parity, empty_out

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _oracle_keys(frags, routing_layer):
    """(id, Q) of each fragment from its full bytes."""
    out = []
    for K, V in frags:
        Kb, Vb = synthetic.to_bits(K), synthetic.to_bits(V)
        out.append((fragment_id(Kb, Vb), norm_key(Kb, routing_layer)))
    return out


def _oracle_order(keys, lengths):
    t_star = min(lengths)
    S = [tail_sum(Q, t_star) for _, Q in keys]
    return sorted(range(len(keys)), key=lambda i: (-S[i], -id_as_int(keys[i][0])))


def _check_all_planes(frags, order, k_out, v_out):
    """Every plane of the render against the oracle: each slot's K rotated by its offset
    (oracle.rotate_k over all layers and heads at once), each slot's V copied."""
    kb, vb = synthetic.to_bits(k_out), synthetic.to_bits(v_out)
    s = 0
    for i in order:
        K, V = frags[i]
        T = K.shape[2]
        want_k = oracle.rotate_k(synthetic.to_bits(K), s, THETA)
        assert assert_k_parity(kb[:, :, s:s + T], want_k, f"K slot@{s}") == 0
        assert np.array_equal(vb[:, :, s:s + T], synthetic.to_bits(V)), f"V slot@{s}"
        del want_k
        s += T
    assert s == kb.shape[2]


def test_q4b_full_size_bench_configuration(ctx):
    w = synthetic.WORKLOADS["q4b"]
    specs = synthetic.fragment_specs(w)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    total = sum(sp.seq_len for sp in specs)
    k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    # the bench's launch configuration: one cm_ingest_render call, replicas A (fragments 0,
    # 1) and B (2, 3), A rendered with the render beside the content address
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    res, n, order_ids, overlapped = cm.cm_ingest_render(
        [A.handle, A.handle, B.handle, B.handle],
        [cm.fragment_from_tensors(K, V) for K, V in frags], A.handle, k_out.data_ptr(),
        v_out.data_ptr(), total)
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    ctx.check()
    torch.cuda.synchronize()
    assert overlapped
    # 4 x 36,864 level-1 nodes: level 1 in its own kernel, then the levels above it
    assert t["leaf_hash_launches"] == 1 and t["inner_hash_launches"] == 2
    assert t["render_launches"] == 1
    keys = _oracle_keys(frags, w.num_layers // 2)
    assert [fid for fid, _ in res] == [k[0] for k in keys]
    assert [a for _, a in res] == [False] * 4
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert order_ids == [keys[i][0] for i in order]
    assert n == total
    _check_all_planes(frags, order, k_out, v_out)
    # the same merge as separate calls: cm_ingest_many, cm_union, cm_render (the full-SM
    # render after the hash), byte for byte
    A2, B2 = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    res2 = cm.ingest_many([(A2, *frags[0]), (A2, *frags[1]), (B2, *frags[2]), (B2, *frags[3])])
    assert res2 == res
    A2.union(B2)
    k2, v2 = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    n2, order2 = A2.render(k2, v2)
    torch.cuda.synchronize()
    assert n2 == n and order2 == order_ids
    assert torch.equal(k2.view(torch.int16), k_out.view(torch.int16))
    assert torch.equal(v2.view(torch.int16), v_out.view(torch.int16))
    for S in (A, B, A2, B2):
        S.close()


def test_split_tree_top_with_roots_at_levels_one_and_two(ctx):
    # one call whose level-1 nodes are enough for the two-kernel tree top, with a
    # fragment whose root is level 1 and one whose root is level 2 beside a full one
    w = synthetic.WORKLOADS["q4b"]
    big = synthetic.make_fragment_torch(synthetic.fragment_specs(w)[0], w.num_layers,
                                        w.num_kv_heads, w.head_dim, "cuda:0")
    g = torch.Generator(device="cuda:0").manual_seed(1716)
    small = [tuple(torch.randn((1, 1, T, 16), generator=g, device="cuda:0").to(torch.bfloat16)
                   for _ in range(2)) for T in (3, 257)]          # 1 and 17 leaves
    sets = [cm.FragmentSet(ctx) for _ in range(3)]
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    res = cm.ingest_many([(sets[0], *small[0]), (sets[1], *big), (sets[2], *small[1])])
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    assert t["inner_hash_launches"] == 2
    want = [fragment_id(synthetic.to_bits(K), synthetic.to_bits(V)) for K, V in (small[0], big, small[1])]
    assert [fid for fid, _ in res] == want
    for S in sets:
        S.close()


def test_redelivery_fast_path_at_full_size():
    # two q4b fragments, each also delivered as a byte-identical clone in its own buffer,
    # into one set with the re-delivery fast path on: the clones take their originals'
    # ids without being hashed (full 604 MB byte comparisons), and the set and its render
    # are the oracle's
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w = synthetic.WORKLOADS["q4b"]
    specs = synthetic.fragment_specs(w)[:2]
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    clones = [(K.clone(), V.clone()) for K, V in frags]
    c = cm.Context(0, THETA)
    cm.cm_context_set_dedup_by_bytes(c.handle, True)
    S = cm.FragmentSet(c)
    cm.cm_context_kernel_times(c.handle, reset=True)
    cm.cm_context_set_timing(c.handle, True)
    res = S.ingest_batch([frags[0], clones[1], clones[0], frags[1]])
    cm.cm_context_set_timing(c.handle, False)
    t = cm.cm_context_kernel_times(c.handle, reset=True)
    assert [a for _, a in res] == [False, False, True, True]
    assert t["leaf_hash_fragments"] == 2           # the first delivery of each fragment only
    keys = _oracle_keys(frags, w.num_layers // 2)
    assert [fid for fid, _ in res] == [keys[0][0], keys[1][0], keys[0][0], keys[1][0]]
    total = sum(sp.seq_len for sp in specs)
    k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    n, order_ids = S.render(k_out, v_out)
    torch.cuda.synchronize()
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert n == total and order_ids == [keys[i][0] for i in order]
    _check_all_planes(frags, order, k_out, v_out)
    S.close()
    c.close()


@pytest.mark.parametrize("request_index", [0, 1])
def test_serving_requests_with_redelivery(ctx, request_index):
    w = synthetic.WORKLOADS["serve"]
    specs = synthetic.fragment_specs(w, request_index)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    sched = synthetic.delivery_schedule(w, request_index)
    msgs = [(frags[i][0].clone(), frags[i][1].clone()) for i in sched]
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(msgs)
    seen = set()
    for (fid, absorbed), i in zip(res, sched):
        assert absorbed == (i in seen)
        seen.add(i)
    assert len(S) == len(specs)
    total = sum(sp.seq_len for sp in specs)
    k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    n, order_ids = S.render(k_out, v_out)
    torch.cuda.synchronize()
    keys = _oracle_keys(frags, w.num_layers // 2)
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert order_ids == [keys[i][0] for i in order] and n == total
    _check_all_planes(frags, order, k_out, v_out)
    S.close()


def test_arity_batch_matches_sequential_ingest_and_oracle(ctx):
    w = synthetic.WORKLOADS["q17_arity"]
    specs = synthetic.fragment_specs(w)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    sched = synthetic.delivery_schedule(w)
    assert len(sched) == 8
    msgs = [(frags[i][0].clone(), frags[i][1].clone()) for i in sched]
    S1 = cm.FragmentSet(ctx)
    batch = S1.ingest_batch(msgs)
    S2 = cm.FragmentSet(ctx)
    seq = [S2.ingest(K, V) for K, V in msgs]
    assert batch == seq
    assert sum(a for _, a in batch) == 3 and len(S1) == 5
    keys = _oracle_keys(frags, w.num_layers // 2)
    assert sorted(S1.ids()) == sorted(k[0] for k in keys)
    total = sum(sp.seq_len for sp in specs)
    outs = []
    for S in (S1, S2):
        k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
        n, order_ids = S.render(k_out, v_out)
        outs.append((k_out, v_out, order_ids))
    torch.cuda.synchronize()
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert outs[0][2] == [keys[i][0] for i in order]
    _check_all_planes(frags, order, outs[0][0], outs[0][1])
    S1.close()
    S2.close()


def test_arity_fused_with_duplicates_matches_the_oracle(ctx):
    # the arity merge through cm_ingest_render: 8 messages (3 byte-duplicates, in buffers
    # of their own) into two replicas; the duplicates are taken for their originals, the
    # render overlaps the content address and stands; every plane against the oracle
    w = synthetic.WORKLOADS["q17_arity"]
    specs = synthetic.fragment_specs(w)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    sched = synthetic.delivery_schedule(w)
    seen, msgs = set(), []
    for i in sched:
        msgs.append(frags[i] if i not in seen else (frags[i][0].clone(), frags[i][1].clone()))
        seen.add(i)
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    half = len(msgs) // 2
    total = sum(sp.seq_len for sp in specs)
    k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    res, n, order_ids, overlapped = cm.cm_ingest_render(
        [A.handle] * half + [B.handle] * (len(msgs) - half),
        [cm.fragment_from_tensors(K, V) for K, V in msgs], A.handle, k_out.data_ptr(),
        v_out.data_ptr(), total)
    torch.cuda.synchronize()
    assert overlapped and n == total and len(A) == 5
    keys = _oracle_keys(frags, w.num_layers // 2)
    assert [r[0] for r in res] == [keys[i][0] for i in sched]
    # absorbed: an earlier message of the same fragment went to the same replica
    dest = [0] * half + [1] * (len(msgs) - half)
    assert [r[1] for r in res] == [any(sched[j] == sched[i] and dest[j] == dest[i] for j in range(i))
                                   for i in range(len(msgs))]
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert order_ids == [keys[i][0] for i in order]
    _check_all_planes(frags, order, k_out, v_out)
    A.close()
    B.close()


def test_arity_all_120_orders_render_identically_at_full_length(ctx):
    # the arity configuration at its real lengths (T ~ U{256..2048}): every order of the
    # five distinct fragments, as unions of single-fragment sets, renders the same bytes;
    # so do 20 random orders of the eight deliveries (duplicates included)
    w = synthetic.WORKLOADS["q17_arity"]
    specs = synthetic.fragment_specs(w)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    total = sum(sp.seq_len for sp in specs)
    singles = []
    for K, V in frags:
        S = cm.FragmentSet(ctx)
        S.ingest(K, V)
        singles.append(S)
    k0, v0 = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    ref = None
    for perm in itertools.permutations(range(5)):
        U = cm.FragmentSet(ctx)
        for i in perm:
            U.union(singles[i])
        n, order_ids = U.render(k0, v0)
        if ref is None:
            ref = (k0.clone(), v0.clone(), order_ids)
        else:
            assert order_ids == ref[2]
            assert torch.equal(k0.view(torch.int16), ref[0].view(torch.int16))
            assert torch.equal(v0.view(torch.int16), ref[1].view(torch.int16))
        U.close()
    sched = synthetic.delivery_schedule(w)
    msgs = [(frags[i][0].clone(), frags[i][1].clone()) for i in sched]
    rng = np.random.default_rng(120)
    for _ in range(20):
        S = cm.FragmentSet(ctx)
        res = S.ingest_batch([msgs[j] for j in rng.permutation(len(msgs))])
        assert sum(a for _, a in res) == 3 and len(S) == 5
        S.render(k0, v0)
        assert torch.equal(k0.view(torch.int16), ref[0].view(torch.int16))
        assert torch.equal(v0.view(torch.int16), ref[1].view(torch.int16))
        S.close()
    keys = _oracle_keys(frags, w.num_layers // 2)
    order = _oracle_order(keys, [sp.seq_len for sp in specs])
    assert ref[2] == [keys[i][0] for i in order]
    _check_all_planes(frags, order, ref[0], ref[1])
    for S in singles:
        S.close()


def test_integer_alu_probe_is_plausible(ctx):
    # the xor chains run on the integer ALU pipe (64 lanes per SM per clock on this
    # part); the compression rate cannot exceed it by more than timing noise
    xor3, comp = cm.cm_measure_int_alu(0)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert sms * 64 * 0.5e9 / 1e12 < xor3 < sms * 64 * 3.0e9 / 1e12
    assert 0.5 * xor3 < comp < 1.05 * xor3


def test_kernel_timing_counts_every_launch(ctx):
    w, L, H, d = None, 4, 2, 64
    g = torch.Generator(device="cuda:0").manual_seed(5)
    frags = [(torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16),
              torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
             for T in (300, 40, 2100)]
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    k_out, v_out = empty_out(L, H, S.seq_len(), d)
    S.render(k_out, v_out)
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    assert t["leaf_hash_launches"] == 1 and t["leaf_hash_fragments"] == 3   # one grouped launch
    assert t["inner_hash_launches"] == 1            # few level-1 nodes: one tree-top kernel
    assert t["render_launches"] == 1
    assert t["aux_launches"] == 1                  # the ingest's result readback
    assert t["leaf_hash_ms"] > 0 and t["render_ms"] > 0
    S.close()
