"""Parity cases run against the bounds-checked build of the library (libcm_bounds.so,
named by the environment variable CM_LIBRARY; started by test_gpu_bounds.py).

Every global access of the render and content-address kernels is checked against the
buffer it belongs to in that build. The cases below cover every kernel path (both render
widths, contiguous, paged with power-of-two and other block sizes, both tree-top schemes,
the allocation-free path, the re-delivery comparison, BagMerge, the incremental render and
both renders that run beside the leaf hash in cm_ingest_render);
their results are checked against the oracle or against each other, and the violation
count must stay 0. A last case renders into a paged cache whose block table holds a
negative entry, an input the host does not check: the bounds-checked build must count it
(the writes go to block 0 instead). Prints one JSON line."""
import json
import os
import sys

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import oracle  # noqa: E402
import paper_2607_01308_gb300 as cm  # noqa: E402
import synthetic  # noqa: E402
from parity_util import THETA, assert_k_parity, empty_out, oracle_fragment  # noqa: E402

DEV = "cuda:0"


def frags_of(seed, L, H, d, lengths, scale=1.0):
    g = torch.Generator(device=DEV).manual_seed(seed)
    return [((torch.randn((L, H, T, d), generator=g, device=DEV) * (scale + 0.1 * i)).to(torch.bfloat16),
             torch.randn((L, H, T, d), generator=g, device=DEV).to(torch.bfloat16))
            for i, T in enumerate(lengths)]


def check_render(ctx, frags, cap_extra=5):
    """Ingest, render with spare capacity, compare ids, order and bytes with the oracle."""
    L, H, _, d = frags[0][0].shape
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(frags)
    refs = [oracle_fragment(K, V) for K, V in frags]
    assert [r[0] for r in res] == [f.fid for f in refs]
    total = S.seq_len()
    k, v = empty_out(L, H, total + cap_extra, d, fill=0x1357)
    n, order = S.render(k, v)
    torch.cuda.synchronize()
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries(refs), THETA)
    assert n == total and order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v[:, :, :n]), V_ref)
    assert assert_k_parity(synthetic.to_bits(k[:, :, :n]), K_ref) == 0
    assert (k.view(torch.int16)[:, :, n:] == 0x1357).all()
    S.close()
    return k[:, :, :n], v[:, :, :n], order


def paged_render(ctx, frags, block_size, table_fn=None):
    """Per-layer pools [L][blocks][bs][H][d]; returns the pools gathered back to [L][H][T][d]."""
    L, H, _, d = frags[0][0].shape
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    total = S.seq_len()
    nb = -(-total // block_size)
    num_blocks = nb + 3
    table = torch.from_numpy(np.random.default_rng(block_size).permutation(num_blocks)[:nb]
                             .astype(np.int32)).to(DEV)
    if table_fn is not None:
        table_fn(table)
    kp = torch.zeros((L, num_blocks, block_size, H, d), dtype=torch.bfloat16, device=DEV)
    vp = torch.zeros_like(kp)
    cache = cm.cm_paged_cache(kp.data_ptr(), vp.data_ptr(), table.data_ptr(), nb, block_size,
                              stride_block=block_size * H * d, stride_layer=num_blocks * block_size * H * d,
                              stride_head=d, stride_token=H * d)
    n, _ = cm.cm_render_paged(S.handle, cache)
    torch.cuda.synchronize()
    pos = torch.arange(total, device=DEV)
    blk = table.long().clamp(min=0)[pos // block_size]
    off = pos % block_size
    S.close()
    return kp[:, blk, off].permute(0, 2, 1, 3), vp[:, blk, off].permute(0, 2, 1, 3)


def main():
    count, enabled = cm.cm_testing_bounds_violations(0)
    # the negative-table case below is only safe in a bounds-checked build
    assert enabled, f"{cm.LIB_PATH} is not a bounds-checked build"
    cases = 0
    ctx = cm.Context(0, THETA)

    # tiny workload, every delivery order; ragged shapes for every head_dim
    w = synthetic.WORKLOADS["tiny"]
    tiny = [synthetic.make_fragment_torch(s, w.num_layers, w.num_kv_heads, w.head_dim, DEV)
            for s in synthetic.fragment_specs(w)]
    check_render(ctx, tiny)
    check_render(ctx, tiny[::-1])
    cases += 2
    for d, lengths in ((16, (1, 129)), (64, (70, 600)), (256, (1, 129, 70)), (512, (3, 40))):
        check_render(ctx, frags_of(100 + d, 3, 2, d, lengths))
        cases += 1

    # 8-warp render CTAs
    cm.cm_context_set_render_warps(ctx.handle, 8)
    check_render(ctx, frags_of(7, 4, 2, 64, (37, 53, 90)))
    cm.cm_context_set_render_warps(ctx.handle, 16)
    cases += 1

    # paged output: power-of-two blocks (per-item bases) and others (per-row lookups)
    fr = frags_of(11, 3, 2, 128, (100, 37, 260))
    kc, vc, _ = check_render(ctx, fr)
    for bs in (16, 64, 12, 1):
        kg, vg = paged_render(ctx, fr, bs)
        assert torch.equal(kg, kc) and torch.equal(vg, vc)
        cases += 1

    # allocation-free content address
    K, V = fr[0]
    L, H, T, d = K.shape
    ref = oracle_fragment(K, V)
    out_id = torch.empty(16, dtype=torch.uint8, device=DEV)
    out_q = torch.empty(T, dtype=torch.int64, device=DEV)
    cm.cm_fragment_id_static(cm.fragment_from_tensors(K, V), out_id.data_ptr(), out_q.data_ptr())
    torch.cuda.synchronize()
    assert bytes(out_id.cpu().numpy().tobytes()) == ref.fid
    assert np.array_equal(out_q.cpu().numpy().view(np.uint64), ref.Q)
    cases += 1

    # 40 fragments: two tree-top calls and two render launches
    many = frags_of(40, 2, 1, 64, [1 + (i * 37) % 50 for i in range(40)], scale=0.5)
    check_render(ctx, many)
    cases += 1

    # the two-kernel tree top (4 x 36,864 level-1 nodes at 4 x 2048 tokens of the q4b shape)
    w = synthetic.WORKLOADS["q4b_t2048"]
    big = [synthetic.make_fragment_torch(s, w.num_layers, w.num_kv_heads, w.head_dim, DEV)
           for s in synthetic.fragment_specs(w)]
    sets = [cm.FragmentSet(ctx) for _ in big]
    res = cm.ingest_many([(S, K, V) for S, (K, V) in zip(sets, big)])
    from oracle.content_address import fragment_id
    assert [r[0] for r in res] == [fragment_id(synthetic.to_bits(K), synthetic.to_bits(V))
                                   for K, V in big]
    for S in sets:
        S.close()
    # the same fragments through cm_ingest_render (1.2 GB of fragments: the 4-warp TMA
    # render beside the leaf hash), byte-equal to the separate calls' render
    total = sum(K.shape[2] for K, _ in big)
    fused_k, fused_v = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    A, B = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    _, n, _, overlapped = cm.cm_ingest_render([A.handle, A.handle, B.handle, B.handle],
                                              [cm.fragment_from_tensors(K, V) for K, V in big],
                                              A.handle, fused_k.data_ptr(), fused_v.data_ptr(), total)
    assert overlapped and n == total
    S = cm.FragmentSet(ctx)
    S.ingest_batch(big)
    seq_k, seq_v = empty_out(w.num_layers, w.num_kv_heads, total, w.head_dim)
    S.render(seq_k, seq_v)
    torch.cuda.synchronize()
    assert torch.equal(fused_k.view(torch.int16), seq_k.view(torch.int16))
    assert torch.equal(fused_v.view(torch.int16), seq_v.view(torch.int16))
    for X in (A, B, S):
        X.close()
    del big, fused_k, fused_v, seq_k, seq_v
    cases += 1
    # a small merge through cm_ingest_render (the register render, one CTA per SM, beside
    # the hash), checked against the oracle
    fs = frags_of(61, 3, 2, 64, (37, 53, 90))
    kc3, vc3, order3 = check_render(ctx, fs)
    A = cm.FragmentSet(ctx)
    k3, v3 = empty_out(3, 2, 180, 64)
    _, n, order, overlapped = cm.cm_ingest_render([A.handle] * 3,
                                                  [cm.fragment_from_tensors(K, V) for K, V in fs],
                                                  A.handle, k3.data_ptr(), v3.data_ptr(), 180)
    torch.cuda.synchronize()
    assert overlapped and n == 180 and order == order3
    assert torch.equal(k3, kc3) and torch.equal(v3, vc3)
    A.close()
    cases += 1

    # re-delivery fast path: clones take their originals' ids without being hashed
    c2 = cm.Context(0, THETA)
    cm.cm_context_set_dedup_by_bytes(c2.handle, True)
    A, B = frags_of(21, 3, 2, 64, (50, 50))
    S = cm.FragmentSet(c2)
    res = S.ingest_batch([A, (B[0].clone(), B[1].clone()), (A[0].clone(), A[1].clone()), B])
    assert [a for _, a in res] == [False, False, True, True]
    assert res[2][0] == res[0][0] == oracle_fragment(*A).fid
    S.close()
    c2.close()
    cases += 1

    # BagMerge in a caller-given order, and the incremental render
    fb = frags_of(31, 2, 2, 64, (20, 33))
    L, H, _, d = fb[0][0].shape
    kb, vb = empty_out(L, H, 53, d)
    n = cm.cm_bagmerge(ctx.handle, [cm.fragment_from_tensors(K, V) for K, V in fb],
                       kb.data_ptr(), vb.data_ptr(), 53)
    torch.cuda.synchronize()
    assert n == 53
    S = cm.FragmentSet(ctx)
    S.ingest_batch(fb[:1])
    ki, vi = empty_out(L, H, 53, d)
    _, order = S.render(ki, vi)
    S.ingest_batch(fb[1:])
    S.render_incremental(ki, vi, order)
    torch.cuda.synchronize()
    kf, vf, _ = check_render(ctx, fb, cap_extra=0)
    assert torch.equal(ki, kf) and torch.equal(vi, vf)
    S.close()
    cases += 2

    # several sets in shared render launches (per-slot outputs of different capacities)
    sa, sb = cm.FragmentSet(ctx), cm.FragmentSet(ctx)
    fa, fb2 = frags_of(51, 2, 2, 64, (30, 17)), frags_of(52, 2, 2, 64, (9, 40, 2))
    cm.ingest_many([(sa, *f) for f in fa] + [(sb, *f) for f in fb2])
    outs = [empty_out(2, 2, sa.seq_len() + 3, 64), empty_out(2, 2, sb.seq_len(), 64)]
    ns = cm.render_many([(sa, *outs[0]), (sb, *outs[1])])
    torch.cuda.synchronize()
    for S, f, (k, v), n in ((sa, fa, outs[0], ns[0]), (sb, fb2, outs[1], ns[1])):
        kr, vr, _ = check_render(ctx, f, cap_extra=0)
        assert n == kr.shape[2]
        assert torch.equal(k[:, :, :n], kr) and torch.equal(v[:, :, :n], vr)
        S.close()
    cases += 1

    # seeded random merges over the accepted shape space, and paged renders of random
    # block sizes (the generator of test_gpu_random.py)
    from test_gpu_random import _case
    for seed in range(10):
        frags, deliveries, _ = _case(700 + seed)
        check_render(ctx, [frags[i] for i in sorted(set(deliveries))], cap_extra=int(seed % 4))
        cases += 1
    for seed, bs in zip(range(6), (1, 3, 8, 17, 64, 128)):
        frags, _, _ = _case(800 + seed)
        kc2, vc2, _ = check_render(ctx, frags, cap_extra=0)
        kg, vg = paged_render(ctx, frags, bs)
        assert torch.equal(kg, kc2) and torch.equal(vg, vc2)
        cases += 1

    clean, _ = cm.cm_testing_bounds_violations(0)

    # positive control: a negative block-table entry must be counted
    def poison(table):
        table[1] = -1
    paged_render(ctx, fr, 16, poison)
    caught, _ = cm.cm_testing_bounds_violations(0)
    ctx.check()
    # the context still renders correctly, with nothing counted
    kg, vg = paged_render(ctx, fr, 16)
    assert torch.equal(kg, kc) and torch.equal(vg, vc)
    after, _ = cm.cm_testing_bounds_violations(0)
    ctx.close()
    print(json.dumps({"enabled": enabled, "violations": clean, "cases": cases,
                      "negative_table_entry_violations": caught, "violations_after": after}))


if __name__ == "__main__":
    main()
