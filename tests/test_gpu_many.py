"""GPU parity of the calls that serve several sets at once and of the replica-exchange
queries: cm_ingest_many, cm_render_many, cm_set_contains, cm_set_leq.

Every rendered set is compared with the CPU oracle's Render of the same set (V and
order bit-exact, K within 1 ulp with 0 non-exact elements) and with the bytes a
per-set cm_render writes; memberships and the inclusion order with the oracle's set.
"""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")

CANARY = 0x5A5A


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _fragments(seed, lengths, L, H, d):
    g = torch.Generator(device="cuda:0").manual_seed(seed)
    out = []
    for i, T in enumerate(lengths):
        K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.5 + 0.07 * i)).to(torch.bfloat16)
        V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
        out.append((K, V))
    return out


def _check_against_oracle(frags, k_out, v_out, total):
    ref = oracle.from_deliveries([oracle_fragment(K, V) for K, V in frags])
    kb, vb = synthetic.to_bits(k_out), synthetic.to_bits(v_out)
    if total:
        K_ref, V_ref, _ = oracle.render(ref, THETA)
        assert np.array_equal(vb[:, :, :total], V_ref)
        assert assert_k_parity(kb[:, :, :total], K_ref) == 0
    assert (kb[:, :, total:] == CANARY).all() and (vb[:, :, total:] == CANARY).all()


@pytest.mark.parametrize("d,num_sets", [(64, 16), (512, 4)])
def test_render_many_matches_oracle_and_per_set_render(ctx, d, num_sets):
    # 16 sets of up to 4 fragments (40 slots) at d = 64 cross the 32-slot launch limit; at d = 512
    # the (cos, sin) table allows 7 slots per launch, so 4 sets of 3 need two launches
    L, H = 2, 2
    rng = np.random.default_rng(d)
    sets, frag_lists, outs = [], [], []
    for i in range(num_sets):
        nf = 0 if i == 1 else (3 if d == 512 else int(rng.integers(1, 5)))   # set 1 is empty
        lengths = [int(x) for x in rng.integers(1, 91, size=nf)]
        frags = _fragments(1000 * d + i, lengths, L, H, d)
        S = cm.FragmentSet(ctx)
        if frags:
            S.ingest_batch(frags)
        total = S.seq_len()
        k, v = empty_out(L, H, total + 5, d, fill=CANARY)
        sets.append(S)
        frag_lists.append(frags)
        outs.append((k, v))
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    lens = cm.render_many([(S, k, v) for S, (k, v) in zip(sets, outs)])
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    torch.cuda.synchronize()
    slots = sum(len(f) for f in frag_lists)
    per_launch = 32 if d == 64 else 7
    assert t["render_launches"] == -(-slots // per_launch)
    for S, frags, (k, v), n in zip(sets, frag_lists, outs, lens):
        assert n == S.seq_len()
        _check_against_oracle(frags, k, v, n)
        if n:
            k1, v1 = empty_out(L, H, n + 5, d, fill=CANARY)
            S.render(k1, v1)
            torch.cuda.synchronize()
            assert torch.equal(k1.view(torch.int16), k.view(torch.int16))
            assert torch.equal(v1.view(torch.int16), v.view(torch.int16))
    for S in sets:
        S.close()


def test_render_many_of_nothing_and_of_empty_sets(ctx):
    assert cm.cm_render_many([]) == []
    S = cm.FragmentSet(ctx)
    assert cm.render_many([(S, None, None), (S, None, None)]) == [0, 0]
    S.close()


def test_ingest_many_equals_sequential_ingest(ctx):
    # three sets; deliveries interleave across them, re-deliver within a set (absorbed)
    # and deliver one fragment to two sets (absorbed in neither: each set is its own state)
    L, H, d = 3, 2, 128
    frags = _fragments(77, [5, 40, 17, 1, 64], L, H, d)
    plan = [(0, 0), (1, 1), (0, 2), (2, 0), (0, 0), (1, 3), (2, 4), (1, 1), (2, 0), (0, 4)]
    sets = [cm.FragmentSet(ctx) for _ in range(3)]
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    res = cm.ingest_many([(sets[s], *frags[f]) for s, f in plan])
    cm.cm_context_set_timing(ctx.handle, False)
    t = cm.cm_context_kernel_times(ctx.handle, reset=True)
    assert t["leaf_hash_launches"] == 1 and t["inner_hash_launches"] == 1
    assert t["leaf_hash_fragments"] == len(plan)
    ref = [oracle_fragment(K, V) for K, V in frags]
    ref_sets = [oracle.FragmentSet() for _ in range(3)]
    for (s, f), (fid, absorbed) in zip(plan, res):
        assert fid == ref[f].fid
        assert absorbed == (ref[f].fid in ref_sets[s])
        ref_sets[s] = oracle.ingest(ref_sets[s], ref[f])
    for S, R in zip(sets, ref_sets):
        assert S.ids() == R.ids()
    # the same deliveries through cm_ingest one at a time give the same sets
    seq = [cm.FragmentSet(ctx) for _ in range(3)]
    for s, f in plan:
        seq[s].ingest(*frags[f])
    assert [S.ids() for S in seq] == [S.ids() for S in sets]
    for S in sets + seq:
        S.close()


def test_ingest_many_shapes_and_errors(ctx):
    a = _fragments(5, [9, 12], 2, 2, 64)
    b = _fragments(6, [7], 3, 1, 32)
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    # sets of different shapes in one call
    res = cm.ingest_many([(A, *a[0]), (B, *b[0]), (A, *a[1])])
    assert [r[1] for r in res] == [False, False, False]
    assert len(A) == 2 and len(B) == 1
    # a delivery whose shape differs from its set's: nothing of the call is inserted
    c = _fragments(7, [4], 2, 2, 64)
    with pytest.raises(cm.CMError) as e:
        cm.ingest_many([(A, *c[0]), (B, *a[0])])
    assert e.value.status == cm.Status.ERR_SHAPE_MISMATCH
    assert len(A) == 2 and len(B) == 1
    # sets of two contexts in one call
    ctx2 = cm.Context(0, THETA)
    C = cm.FragmentSet(ctx2)
    with pytest.raises(cm.CMError) as e:
        cm.ingest_many([(A, *c[0]), (C, *c[0])])
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    assert len(A) == 2 and len(C) == 0
    with pytest.raises(cm.CMError) as e:
        cm.cm_ingest_many([A.handle, 0], [cm.fragment_from_tensors(*c[0])] * 2)
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    C.close()
    ctx2.close()
    A.close()
    B.close()


def test_render_many_errors_launch_nothing(ctx):
    L, H, d = 2, 2, 64
    A, B, D = cm.FragmentSet(ctx), cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    A.ingest_batch(_fragments(11, [8, 9], L, H, d))
    B.ingest_batch(_fragments(12, [10], L, H, d))
    D.ingest_batch(_fragments(13, [6], L, H, 32))
    ka, va = empty_out(L, H, 17, d, fill=CANARY)
    kb, vb = empty_out(L, H, 9, d, fill=CANARY)          # one token short
    with pytest.raises(cm.CMError) as e:
        cm.render_many([(A, ka, va), (B, kb, vb)])
    assert e.value.status == cm.Status.ERR_CAPACITY
    torch.cuda.synchronize()
    assert (ka.view(torch.int16) == CANARY).all()      # job 0 was not rendered either
    kd, vd = empty_out(L, H, 6, 32)
    with pytest.raises(cm.CMError) as e:
        cm.render_many([(A, ka, va), (D, kd, vd)])
    assert e.value.status == cm.Status.ERR_SHAPE_MISMATCH
    with pytest.raises(cm.CMError) as e:
        cm.cm_render_many([cm.cm_render_job(0, ka.data_ptr(), va.data_ptr(), 17)])
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    ctx2 = cm.Context(0, THETA)
    E = cm.FragmentSet(ctx2)
    E.ingest_batch(_fragments(14, [3], L, H, d))
    ke, ve = empty_out(L, H, 3, d)
    with pytest.raises(cm.CMError) as e:
        cm.render_many([(A, ka, va), (E, ke, ve)])
    assert e.value.status == cm.Status.ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert (ka.view(torch.int16) == CANARY).all()
    for S in (A, B, D, E):
        S.close()
    ctx2.close()


def test_replica_exchange_by_ids(ctx):
    # Section 4.4: replicas A and B exchange ids, then ship only the fragments the other
    # lacks; both end at the union, render identical bytes, and the inclusion order
    # holds at every step
    L, H, d = 2, 2, 64
    frags = _fragments(21, [11, 30, 7, 19, 25], L, H, d)
    ref = [oracle_fragment(K, V) for K, V in frags]
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    A.ingest_batch([frags[i] for i in (0, 1, 2)])
    B.ingest_batch([frags[i] for i in (2, 3, 4)])
    RA = oracle.from_deliveries([ref[i] for i in (0, 1, 2)])
    RB = oracle.from_deliveries([ref[i] for i in (2, 3, 4)])
    assert (A <= B) == RA.leq(RB) == False  # noqa: E712
    assert (A <= A) and (B <= B)
    by_id = {r.fid: kv for r, kv in zip(ref, frags)}
    b_ids = B.ids()
    present = A.contains(b_ids)
    assert present == [fid in RA for fid in b_ids]
    A.ingest_batch([by_id[fid] for fid, p in zip(b_ids, present) if not p])
    a_ids = A.ids()
    present = B.contains(a_ids)
    assert present == [fid in RB for fid in a_ids]
    B.ingest_batch([by_id[fid] for fid, p in zip(a_ids, present) if not p])
    RU = oracle.union(RA, RB)
    assert A.ids() == B.ids() == RU.ids()
    assert (A <= B) and (B <= A)
    total = A.seq_len()
    outs = [empty_out(L, H, total, d) for _ in range(2)]
    cm.render_many([(A, *outs[0]), (B, *outs[1])])
    torch.cuda.synchronize()
    assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
    assert torch.equal(outs[0][1].view(torch.int16), outs[1][1].view(torch.int16))
    K_ref, V_ref, _ = oracle.render(RU, THETA)
    assert np.array_equal(synthetic.to_bits(outs[0][1]), V_ref)
    assert assert_k_parity(synthetic.to_bits(outs[0][0]), K_ref) == 0
    empty = cm.FragmentSet(ctx)
    assert (empty <= A) and not (A <= empty)
    assert A.contains([]) == []
    for S in (A, B, empty):
        S.close()


def test_eight_warp_render_writes_the_same_bytes(ctx):
    # cm_context_set_render_warps(8) halves the render CTA; every layout must come out
    # byte-identical to the default 16-warp render (and so to the oracle)
    ctx8 = cm.Context(0, THETA)
    cm.cm_context_set_render_warps(ctx8.handle, 8)
    for bad in (0, 4, 12, 32):
        with pytest.raises(cm.CMError) as e:
            cm.cm_context_set_render_warps(ctx8.handle, bad)
        assert e.value.status == cm.Status.ERR_INVALID_ARG
    for d in (16, 64, 128, 512):
        L, H = 3, 2
        frags = _fragments(8000 + d, [1, 129, 70, 600], L, H, d)
        outs = []
        for c in (ctx, ctx8):
            S = cm.FragmentSet(c)
            S.ingest_batch(frags)
            k, v = empty_out(L, H, S.seq_len() + 3, d, fill=CANARY)
            S.render(k, v)
            torch.cuda.synchronize()
            outs.append((k, v))
            S.close()
        assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
        assert torch.equal(outs[0][1].view(torch.int16), outs[1][1].view(torch.int16))
        if d == 128:
            _check_against_oracle(frags, outs[1][0], outs[1][1], sum([1, 129, 70, 600]))
    # paged output and BagMerge through the 8-warp kernel
    L, H, d, bs = 2, 2, 64, 16
    frags = _fragments(8100, [37, 200, 5], L, H, d)
    total = sum(f[0].shape[2] for f in frags)
    nblk = -(-total // bs)
    table = torch.randperm(nblk, generator=torch.Generator().manual_seed(1)).to(torch.int32).cuda()
    pools = []
    for c in (ctx, ctx8):
        S = cm.FragmentSet(c)
        S.ingest_batch(frags)
        kp = torch.zeros((L, nblk, bs, H, d), dtype=torch.bfloat16, device="cuda:0")
        vp = torch.zeros_like(kp)
        cache = cm.cm_paged_cache(kp.data_ptr(), vp.data_ptr(), table.data_ptr(), nblk, bs,
                                  stride_block=bs * H * d, stride_layer=nblk * bs * H * d,
                                  stride_head=d, stride_token=H * d)
        cm.cm_render_paged(S.handle, cache)
        torch.cuda.synchronize()
        pools.append((kp, vp))
        S.close()
    assert torch.equal(pools[0][0].view(torch.int16), pools[1][0].view(torch.int16))
    assert torch.equal(pools[0][1].view(torch.int16), pools[1][1].view(torch.int16))
    seq = frags + frags[:1]
    n_tok = sum(f[0].shape[2] for f in seq)
    bag = []
    for c in (ctx, ctx8):
        kb, vb = empty_out(L, H, n_tok, d)
        c.bagmerge(seq, kb, vb)
        torch.cuda.synchronize()
        bag.append((kb, vb))
    assert torch.equal(bag[0][0].view(torch.int16), bag[1][0].view(torch.int16))
    assert torch.equal(bag[0][1].view(torch.int16), bag[1][1].view(torch.int16))
    ctx8.close()


def test_overlapped_groups_match_the_oracle():
    # the serving loop's overlap: group g renders (8-warp CTAs) on the compute stream while
    # group g + 1 is hashed on a second stream; every request's cache equals the oracle's
    c = cm.Context(0, THETA)
    cm.cm_context_set_render_warps(c.handle, 8)
    L, H, d = 8, 4, 128
    rng = np.random.default_rng(31)
    reqs = []
    for r in range(9):
        frags = _fragments(700 + r, [int(t) for t in rng.integers(150, 600, size=3)], L, H, d)
        deliveries = frags + ([frags[int(rng.integers(0, 3))]] if r % 2 else [])
        reqs.append((frags, deliveries))
    outs = [empty_out(L, H, sum(K.shape[2] for K, _ in f), d, fill=CANARY) for f, _ in reqs]
    stream = torch.cuda.current_stream()
    s_hash = torch.cuda.Stream()
    groups = [list(range(g0, g0 + 3)) for g0 in range(0, 9, 3)]

    def ingest(group):
        sets = [cm.FragmentSet(c) for _ in group]
        cm.ingest_many([(S, K, V) for S, r in zip(sets, group) for K, V in reqs[r][1]], s_hash)
        return sets

    s_hash.wait_stream(stream)
    sets = ingest(groups[0])
    lens, held = [], []
    for gi, group in enumerate(groups):
        stream.wait_stream(s_hash)
        lens += cm.render_many([(S, *outs[r]) for S, r in zip(sets, group)], stream)
        held += sets
        if gi + 1 < len(groups):
            sets = ingest(groups[gi + 1])
    stream.wait_stream(s_hash)
    torch.cuda.synchronize()
    for r, (frags, _) in enumerate(reqs):
        refs = [oracle_fragment(K, V) for K, V in frags]
        K_ref, V_ref, _ = oracle.render(oracle.from_deliveries(refs), THETA)
        k, v = outs[r]
        assert lens[r] == K_ref.shape[2]
        assert np.array_equal(synthetic.to_bits(v), V_ref)
        assert assert_k_parity(synthetic.to_bits(k), K_ref) == 0
    for S in held:
        S.close()
    c.close()
