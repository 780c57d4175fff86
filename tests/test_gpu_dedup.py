"""The re-delivery fast path (cm_context_set_dedup_by_bytes): a delivery byte-identical
to a fragment of known id takes that id without being hashed. Every result (ids,
absorption, set contents, rendered bytes) must equal the result with the path off, and
the ids must equal the oracle's; near-duplicates that differ in one bit must be hashed
and get their own ids."""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


@pytest.fixture(scope="module")
def ctxs():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    off = cm.Context(0, THETA)
    on = cm.Context(0, THETA)
    cm.cm_context_set_dedup_by_bytes(on.handle, True)
    yield off, on
    off.close()
    on.close()


def _frags(seed, lengths, L=3, H=2, d=64):
    g = torch.Generator(device="cuda:0").manual_seed(seed)
    return [((torch.randn((L, H, T, d), generator=g, device="cuda:0") * (0.6 + 0.1 * i)).to(torch.bfloat16),
             torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16))
            for i, T in enumerate(lengths)]


def _clone(f):
    return f[0].clone(), f[1].clone()


def _flip(f, which, index):
    K, V = _clone(f)
    t = (K if which == "k" else V).view(torch.int16).view(-1)
    t[index] ^= 1
    return K, V


def _timed(ctx, fn):
    cm.cm_context_kernel_times(ctx.handle, reset=True)
    cm.cm_context_set_timing(ctx.handle, True)
    out = fn()
    cm.cm_context_set_timing(ctx.handle, False)
    return out, cm.cm_context_kernel_times(ctx.handle, reset=True)


def test_results_equal_with_the_fast_path_on_and_off(ctxs):
    A, B, C = _frags(900, [50, 50, 30])
    n_elem = A[0].numel()
    clones = [_clone(A) for _ in range(3)]
    near = [_flip(A, "v", -1), _flip(A, "k", 0), _flip(A, "k", n_elem // 2), _flip(A, "v", n_elem // 3)]
    plan = [(0, A), (0, clones[0]), (0, A), (0, near[0]), (0, near[1]), (0, B), (0, near[2]),
            (0, clones[1]), (1, clones[2]), (1, C), (1, B), (1, near[3]), (0, C)]
    results = []
    for ctx in ctxs:
        sets = [cm.FragmentSet(ctx), cm.FragmentSet(ctx)]
        res = cm.ingest_many([(sets[s], *f) for s, f in plan])
        outs = []
        for S in sets:
            k, v = empty_out(3, 2, S.seq_len(), 64)
            S.render(k, v)
            outs.append((k, v))
        torch.cuda.synchronize()
        results.append((res, [S.ids() for S in sets], outs))
        for S in sets:
            S.close()
    (res_off, ids_off, outs_off), (res_on, ids_on, outs_on) = results
    assert res_on == res_off
    assert ids_on == ids_off
    for (k0, v0), (k1, v1) in zip(outs_off, outs_on):
        assert torch.equal(k0.view(torch.int16), k1.view(torch.int16))
        assert torch.equal(v0.view(torch.int16), v1.view(torch.int16))
    # the ids are the oracle's, near-duplicates included
    for (s, f), (fid, _) in zip(plan, res_on):
        assert fid == oracle_fragment(*f).fid
    assert len({fid for fid, _ in res_on}) == 7     # A, B, C and four near-duplicates
    # the rendered union of set 1 (a clone of A, C, B, a near-duplicate) is the oracle's
    ref = oracle.from_deliveries([oracle_fragment(*f) for s, f in plan if s == 1])
    K_ref, V_ref, _ = oracle.render(ref, THETA)
    assert np.array_equal(synthetic.to_bits(outs_on[1][1]), V_ref)
    assert assert_k_parity(synthetic.to_bits(outs_on[1][0]), K_ref) == 0


def test_duplicates_are_not_hashed(ctxs):
    _, on = ctxs
    A, B = _frags(910, [40, 41])
    c1, c2 = _clone(A), _clone(A)
    S = cm.FragmentSet(on)
    res, t = _timed(on, lambda: S.ingest_batch([A, c1, c2, B, A]))
    assert [a for _, a in res] == [False, True, True, False, True]
    assert res[1][0] == res[2][0] == res[4][0] == res[0][0]
    assert t["leaf_hash_fragments"] == 2           # A and B only
    # a later call: a clone of a fragment the set holds is absorbed with no hashing at all
    c3 = _clone(B)
    res2, t2 = _timed(on, lambda: S.ingest_batch([c3]))
    assert res2 == [(res[3][0], True)]
    assert t2["leaf_hash_fragments"] == 0 and t2["leaf_hash_launches"] == 0
    assert t2["inner_hash_launches"] == 0
    # in one call, a clone delivered to another set than its original takes the
    # original's id and norm key: the order of that set's render (which needs the norm
    # key) and its bytes are the oracle's
    U, T = cm.FragmentSet(on), cm.FragmentSet(on)
    res3, t3 = _timed(on, lambda: cm.ingest_many([(U, *B), (T, *_clone(B)), (T, *A)]))
    assert [a for _, a in res3] == [False, False, False]
    assert t3["leaf_hash_fragments"] == 2          # B and A; the clone is not hashed
    kT, vT = empty_out(3, 2, 81, 64)
    n, order = T.render(kT, vT)
    ref = oracle.from_deliveries([oracle_fragment(*B), oracle_fragment(*A)])
    K_ref, V_ref, o_order = oracle.render(ref, THETA)
    torch.cuda.synchronize()
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(vT), V_ref)
    assert assert_k_parity(synthetic.to_bits(kT), K_ref) == 0
    for X in (S, U, T):
        X.close()


def test_fast_path_with_verify_on_hit():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ctx = cm.Context(0, THETA, verify_bytes_on_hit=True)
    cm.cm_context_set_dedup_by_bytes(ctx.handle, True)
    A, = _frags(920, [33])
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch([A, _clone(A)])
    assert [a for _, a in res] == [False, True]
    res2 = S.ingest_batch([_clone(A)])
    assert res2 == [(res[0][0], True)]
    S.close()
    ctx.close()


@pytest.mark.parametrize("seed", range(10))
def test_random_redeliveries_equal_the_path_off(ctxs, seed):
    # seeded random merges (the generator of test_gpu_random.py) with every delivery a
    # separate buffer, re-sent copies in random order and, in every other case, a one-bit
    # near-duplicate of one fragment; spread over one or two ingest calls, then a union
    from test_gpu_random import _case
    off, on = ctxs
    rng = np.random.default_rng(6000 + seed)
    frags, deliveries, _ = _case(400 + seed)
    msgs = [_clone(frags[i]) for i in deliveries]
    if seed % 2:
        K, V = _clone(frags[int(rng.integers(0, len(frags)))])
        K.view(torch.int16).view(-1)[int(rng.integers(0, K.numel()))] ^= 1
        msgs.insert(int(rng.integers(0, len(msgs) + 1)), (K, V))
    cut = int(rng.integers(0, len(msgs) + 1))
    L, H, _, d = frags[0][0].shape
    results = []
    for c in (off, on):
        A, B = cm.FragmentSet(c), cm.FragmentSet(c)
        res = A.ingest_batch(msgs[:cut]) + B.ingest_batch(msgs[cut:])
        B.ingest_batch(msgs[:cut])                 # B re-receives A's deliveries
        A.union(B)
        k, v = empty_out(L, H, A.seq_len(), d)
        n, order = A.render(k, v)
        torch.cuda.synchronize()
        results.append((res, sorted(A.ids()), n, order, synthetic.to_bits(k), synthetic.to_bits(v)))
        A.close()
        B.close()
    (r0, ids0, n0, o0, k0, v0), (r1, ids1, n1, o1, k1, v1) = results
    assert r0 == r1 and ids0 == ids1 and n0 == n1 and o0 == o1
    assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    refs = [oracle_fragment(K, V) for K, V in msgs]
    assert [fid for fid, _ in r0] == [f.fid for f in refs]
    K_ref, V_ref, o_ref = oracle.render(oracle.from_deliveries(refs), THETA)
    assert o0 == [f.fid for f in o_ref] and np.array_equal(v0, V_ref)
    assert assert_k_parity(k0, K_ref) == 0
