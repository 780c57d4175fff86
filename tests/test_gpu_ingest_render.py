"""GPU parity of cm_ingest_render: ingest into several replicas, union into the target and
render, with the render overlapping the content address when the norm-key sums decide
the canonical order (Algorithm 1) on their own.

Every case is compared with the CPU oracle (ids, absorption flags, order and V
bit-exact, K within 1 ulp with 0 non-exact elements) and with the same sequence of
separate calls (cm_ingest_many, cm_union, cm_render) on the library, byte for byte;
the overlapped flag says whether the render started beside the content address stood:
it does for distinct sums and for duplicate deliveries (equal sums, lengths and norm keys
are taken for one fragment, which the ids then confirm); it does not for an exact tie
of the sums between different fragments (the speculative render is replaced once the
ids are known), the re-delivery fast path and an output the render refuses.
"""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, gpu_fragments, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")

CANARY = 0x3C3C


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _fragments(seed, lengths, L=3, H=2, d=64, scales=None):
    g = torch.Generator(device="cuda:0").manual_seed(seed)
    out = []
    for i, T in enumerate(lengths):
        sc = scales[i] if scales else 0.6 + 0.15 * i
        K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * sc).to(torch.bfloat16)
        V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
        out.append((K, V))
    return out


def _fused(ctx, sets, deliveries, target, cap, stream=None):
    """cm_ingest_render into canary-filled outputs; returns (outputs, results)."""
    L, H, _, d = deliveries[0][0].shape if deliveries else (1, 1, 1, 16)
    k, v = empty_out(L, H, cap, d, fill=CANARY)
    fd = [cm.fragment_from_tensors(K, V) for K, V in deliveries]
    res = cm.cm_ingest_render([s.handle for s in sets], fd, target.handle, k.data_ptr(),
                              v.data_ptr(), cap, stream)
    torch.cuda.synchronize()
    return (k, v), res


def _sequence(ctx, sets, deliveries, target, cap):
    """The same steps as separate calls on fresh sets holding the same prior records."""
    L, H, _, d = deliveries[0][0].shape
    k, v = empty_out(L, H, cap, d, fill=CANARY)
    fd = [cm.fragment_from_tensors(K, V) for K, V in deliveries]
    res = cm.cm_ingest_many([s.handle for s in sets], fd)
    for s in dict.fromkeys(sets):
        if s is not target:
            target.union(s)
    n, order = target.render(k, v)
    torch.cuda.synchronize()
    return (k, v), res, n, order


def _check(out, n, union_of, ids_expected=None):
    """Output against the oracle's render of the set made of the fragments `union_of`."""
    ref = oracle.from_deliveries([oracle_fragment(K, V) for K, V in union_of])
    K_ref, V_ref, o_order = oracle.render(ref, THETA)
    kb, vb = synthetic.to_bits(out[0]), synthetic.to_bits(out[1])
    assert n == K_ref.shape[2]
    assert np.array_equal(vb[:, :, :n], V_ref)
    assert assert_k_parity(kb[:, :, :n], K_ref) == 0
    assert (kb[:, :, n:] == CANARY).all() and (vb[:, :, n:] == CANARY).all()
    return [f.fid for f in o_order]


def test_two_replicas_distinct_sums_overlap_and_match_the_oracle(ctx):
    frags = _fragments(11, [37, 129, 70, 600])
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    sets = [A, A, B, B]
    out, (res, n, order, overlapped) = _fused(ctx, sets, frags, A, 900)
    assert overlapped
    assert [a for _, a in res] == [False] * 4
    assert [i for i, _ in res] == [oracle_fragment(K, V).fid for K, V in frags]
    assert order == _check(out, n, frags)
    assert len(A) == 4 and len(B) == 2
    # byte-identical to the separate calls
    A2, B2 = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    out2, res2, n2, order2 = _sequence(ctx, [A2, A2, B2, B2], frags, A2, 900)
    assert res2 == res and n2 == n and order2 == order
    assert torch.equal(out[0].view(torch.int16), out2[0].view(torch.int16))
    assert torch.equal(out[1].view(torch.int16), out2[1].view(torch.int16))
    for s in (A, B, A2, B2):
        s.close()


def test_prior_records_and_other_replicas_join_the_speculation(ctx):
    frags = _fragments(12, [50, 51, 52, 53, 54, 55])
    A, B, C = cm.FragmentSet(ctx), cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    A.ingest_batch(frags[:1])
    B.ingest_batch(frags[1:3])
    # C receives two deliveries, A one, B one; the target is A
    sets = [C, A, B, C]
    out, (res, n, order, overlapped) = _fused(ctx, sets, frags[3:] + frags[:1], A, 400)
    # the last delivery repeats A's record: equal sums, lengths and norm keys, taken for
    # the same fragment, which the ids confirm (A keeps its record)
    assert overlapped
    assert [a for _, a in res] == [False, False, False, False]   # C did not hold it
    assert order == _check(out, n, frags)
    out, (res, n, order, overlapped) = _fused(ctx, [C], frags[3:4], A, 400)
    assert overlapped and res[0][1]                              # absorbed by C
    assert order == _check(out, n, frags)
    for s in (A, B, C):
        s.close()
    # distinct sums with prior records in the target and in another replica
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    A.ingest_batch(frags[:2])
    B.ingest_batch(frags[2:3])
    out, (res, n, order, overlapped) = _fused(ctx, [B, A, B], frags[3:], A, 400)
    assert overlapped
    assert order == _check(out, n, frags)
    assert len(A) == 6 and len(B) == 3
    A.close()
    B.close()


def test_exact_tie_of_the_sums_runs_after_the_ids(ctx):
    # equal K (so equal norm keys and equal sums), different V: taken for one fragment by
    # the speculation, which the ids refute; the order needs the ids, and the target is
    # rendered again after the speculative render
    (K0, V0), (_, V1), (K2, V2) = _fragments(13, [40, 40, 47])
    frags = [(K0, V0), (K0.clone(), V1), (K2, V2)]
    A = cm.FragmentSet(ctx)
    out, (res, n, order, overlapped) = _fused(ctx, [A, A, A], frags, A, 200)
    assert not overlapped
    assert [a for _, a in res] == [False, False, False]
    assert order == _check(out, n, frags)
    # the same with the tie across two replicas and a byte copy of the third fragment
    B, A2 = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    out, (res, n, order, overlapped) = _fused(ctx, [A2, B, B, A2],
                                              frags + [(K2.clone(), V2.clone())], A2, 200)
    assert not overlapped
    assert [a for _, a in res] == [False, False, False, False]   # the copy went to A2
    assert order == _check(out, n, frags)
    for s in (A, B, A2):
        s.close()


def test_duplicate_delivery_is_absorbed(ctx):
    frags = _fragments(14, [33, 66, 99])
    deliveries = frags + [(frags[1][0].clone(), frags[1][1].clone())]
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    # the copy of fragment 1 goes to the replica that already received it: the copy is
    # taken for the same fragment, the render overlaps and stands
    out, (res, n, order, overlapped) = _fused(ctx, [A, B, A, B], deliveries, A, 300)
    assert overlapped
    assert [a for _, a in res] == [False, False, False, True]
    assert order == _check(out, n, frags)
    # byte-equal to the separate calls
    A2, B2 = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    out2, res2, n2, order2 = _sequence(ctx, [A2, B2, A2, B2], deliveries, A2, 300)
    assert res2 == res and n2 == n and order2 == order
    assert torch.equal(out[0].view(torch.int16), out2[0].view(torch.int16))
    assert torch.equal(out[1].view(torch.int16), out2[1].view(torch.int16))
    A2.close()
    B2.close()
    A.close()
    B.close()


def test_redelivery_fast_path_and_refused_output_take_the_sequence(ctx):
    frags = _fragments(15, [20, 21])
    c2 = cm.Context(0, THETA)
    cm.cm_context_set_dedup_by_bytes(c2.handle, True)
    A = cm.FragmentSet(c2)
    out, (res, n, order, overlapped) = _fused(c2, [A, A], frags, A, 64)
    assert not overlapped
    assert order == _check(out, n, frags)
    A.close()
    c2.close()
    # an output too short for the set: the deliveries are ingested, then the render fails
    A = cm.FragmentSet(ctx)
    with pytest.raises(cm.CMError) as e:
        _fused(ctx, [A, A], frags, A, 40)
    assert e.value.status == cm.Status.ERR_CAPACITY
    assert len(A) == 2
    A.close()


def test_shape_mismatch_is_refused_before_any_work(ctx):
    a = _fragments(16, [10], L=2)
    b = _fragments(17, [10], L=3)
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    B.ingest_batch(b)
    with pytest.raises(cm.CMError) as e:
        _fused(ctx, [B, A], a + a, A, 64)
    assert e.value.status == cm.Status.ERR_SHAPE_MISMATCH
    assert len(A) == 0 and len(B) == 1
    A.close()
    B.close()


@pytest.mark.parametrize("workload", ["q17_n2", "q4b_t512", "q4b_t2048"])
def test_model_shaped_merges_overlap_and_match(ctx, workload):
    w, frags, _ = gpu_fragments(workload)
    half = (len(frags) + 1) // 2
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    total = sum(K.shape[2] for K, _ in frags)
    out, (res, n, order, overlapped) = _fused(ctx, [A] * half + [B] * (len(frags) - half),
                                              frags, A, total + 3)
    assert overlapped
    assert order == _check(out, n, frags)
    A2, B2 = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    out2, res2, n2, order2 = _sequence(ctx, [A2] * half + [B2] * (len(frags) - half), frags, A2,
                                       total + 3)
    assert order2 == order
    assert torch.equal(out[0].view(torch.int16), out2[0].view(torch.int16))
    assert torch.equal(out[1].view(torch.int16), out2[1].view(torch.int16))
    for s in (A, B, A2, B2):
        s.close()


def test_side_stream_result_is_ordered_before_later_work_on_the_stream(ctx):
    # a copy enqueued on the caller's stream right after the call sees the finished render
    frags = _fragments(18, [300, 301, 302])
    A = cm.FragmentSet(ctx)
    s = torch.cuda.Stream()
    k, v = empty_out(3, 2, 903, 64, fill=CANARY)
    fd = [cm.fragment_from_tensors(K, V) for K, V in frags]
    with torch.cuda.stream(s):
        _, n, _, overlapped = cm.cm_ingest_render([A.handle] * 3, fd, A.handle, k.data_ptr(),
                                                  v.data_ptr(), 903, s)
        k_copy, v_copy = k.clone(), v.clone()
    s.synchronize()
    assert overlapped
    _check((k_copy, v_copy), n, frags)
    A.close()


def test_overlap_modes_give_the_same_bytes(ctx):
    frags = _fragments(19, [64, 65, 66])
    outs = []
    for mode in (0, 1):
        c = cm.Context(0, THETA)
        cm.cm_context_set_overlap(c.handle, mode)
        A = cm.FragmentSet(c)
        out, (res, n, order, overlapped) = _fused(c, [A] * 3, frags, A, 200)
        assert overlapped == (mode == 1)
        outs.append((out, order))
        A.close()
        c.close()
    assert outs[1][1] == outs[0][1]
    assert torch.equal(outs[1][0][0].view(torch.int16), outs[0][0][0].view(torch.int16))
    assert torch.equal(outs[1][0][1].view(torch.int16), outs[0][0][1].view(torch.int16))
    _check(outs[0][0], sum(K.shape[2] for K, _ in frags), frags)
    for bad in (2, -1):
        with pytest.raises(cm.CMError):
            cm.cm_context_set_overlap(ctx.handle, bad)
