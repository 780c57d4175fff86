"""Randomised GPU parity: seeded random merges over the whole shape space the library
accepts (layers, heads, every head_dim, 1..5 fragments of ragged lengths, lengths at and
next to work-item boundaries, byte-identical re-deliveries in random order, spare output
capacity), each compared with the CPU oracle: ids, absorption, order and V bit-exact, K
within 1 ulp and bit-exact in count, and the rows beyond the merged length untouched."""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")

HEAD_DIMS = (16, 32, 64, 128, 256, 512)


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _case(seed):
    rng = np.random.default_rng(1000 + seed)
    L = int(rng.integers(1, 7))
    H = int(rng.integers(1, 5))
    d = int(rng.choice(HEAD_DIMS))
    rows_per_item = 4096 // (2 * d)
    n = int(rng.integers(1, 6))
    lengths = []
    for _ in range(n):
        if rng.random() < 0.4:   # at or next to a work-item boundary
            lengths.append(max(1, rows_per_item * int(rng.integers(1, 5)) + int(rng.integers(-1, 2))))
        else:   # up to 700 tokens at d = 64, fewer for wider heads (the oracle's cost)
            lengths.append(int(rng.integers(1, max(9, 700 * 64 // d))))
    g = torch.Generator(device="cuda:0").manual_seed(2000 + seed)
    frags = [((torch.randn((L, H, T, d), generator=g, device="cuda:0") * float(rng.uniform(0.3, 3.0)))
              .to(torch.bfloat16),
              (torch.randn((L, H, T, d), generator=g, device="cuda:0") * float(rng.uniform(0.3, 3.0)))
              .to(torch.bfloat16)) for T in lengths]
    deliveries = list(range(n)) + [int(i) for i in rng.integers(0, n, size=int(rng.integers(0, 3)))]
    rng.shuffle(deliveries)
    extra = int(rng.integers(0, 40))
    return frags, deliveries, extra


@pytest.mark.parametrize("seed", range(25))
def test_random_merge_matches_oracle(ctx, seed):
    frags, deliveries, extra = _case(seed)
    L, H, _, d = frags[0][0].shape
    msgs = [(frags[i][0].clone(), frags[i][1].clone()) for i in deliveries]
    S = cm.FragmentSet(ctx)
    res = S.ingest_batch(msgs)
    refs = [oracle_fragment(K, V) for K, V in frags]
    seen = set()
    for (fid, absorbed), i in zip(res, deliveries):
        assert fid == refs[i].fid
        assert absorbed == (i in seen)
        seen.add(i)
    total = S.seq_len()
    k, v = empty_out(L, H, total + extra, d, fill=0x2468)
    n, order = S.render(k, v)
    torch.cuda.synchronize()
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries([refs[i] for i in deliveries]), THETA)
    assert n == total == K_ref.shape[2]
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v[:, :, :n]), V_ref)
    assert assert_k_parity(synthetic.to_bits(k[:, :, :n]), K_ref) == 0
    assert (k.view(torch.int16)[:, :, n:] == 0x2468).all() and (v.view(torch.int16)[:, :, n:] == 0x2468).all()
    S.close()


@pytest.mark.parametrize("seed", range(12))
def test_random_paged_render_matches_contiguous(ctx, seed):
    frags, deliveries, _ = _case(100 + seed)
    L, H, _, d = frags[0][0].shape
    rng = np.random.default_rng(3000 + seed)
    bs = int(rng.choice((1, 3, 8, 16, 17, 64, 128)))
    layout = "per_layer" if rng.random() < 0.5 else "block_major"
    S = cm.FragmentSet(ctx)
    S.ingest_batch([frags[i] for i in deliveries])
    total = S.seq_len()
    k, v = empty_out(L, H, total, d)
    n, order = S.render(k, v)
    nb = -(-total // bs)
    num_blocks = nb + int(rng.integers(1, 5))
    table = torch.from_numpy(rng.permutation(num_blocks)[:nb].astype(np.int32)).to("cuda:0")
    if layout == "per_layer":          # [L][num_blocks][bs][H][d]
        shape = (L, num_blocks, bs, H, d)
        strides = dict(stride_layer=num_blocks * bs * H * d, stride_block=bs * H * d,
                       stride_token=H * d, stride_head=d)
    else:                              # [num_blocks][L][H][bs][d]
        shape = (num_blocks, L, H, bs, d)
        strides = dict(stride_block=L * H * bs * d, stride_layer=H * bs * d,
                       stride_head=bs * d, stride_token=d)
    kp = torch.full(shape, 0x1357, dtype=torch.int16, device="cuda:0").view(torch.bfloat16)
    vp = torch.full(shape, 0x1357, dtype=torch.int16, device="cuda:0").view(torch.bfloat16)
    cache = cm.cm_paged_cache(kp.data_ptr(), vp.data_ptr(), table.data_ptr(), nb, bs, **strides)
    n2, order2 = cm.cm_render_paged(S.handle, cache)
    torch.cuda.synchronize()
    assert n2 == n and order2 == order
    pos = torch.arange(total, device="cuda:0")
    blk = table.long()[pos // bs]
    off = pos % bs
    if layout == "per_layer":
        kg, vg = kp[:, blk, off].permute(0, 2, 1, 3), vp[:, blk, off].permute(0, 2, 1, 3)
    else:
        kg, vg = kp[blk, :, :, off].permute(1, 2, 0, 3), vp[blk, :, :, off].permute(1, 2, 0, 3)
    assert torch.equal(kg, k) and torch.equal(vg, v)
    # and the gathered paged result against the oracle directly
    refs = [oracle_fragment(K, V) for K, V in frags]
    K_ref, V_ref, o_order = oracle.render(oracle.from_deliveries([refs[i] for i in deliveries]), THETA)
    assert order2 == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(vg), V_ref)
    assert assert_k_parity(synthetic.to_bits(kg), K_ref) == 0
    spare = [b for b in range(num_blocks) if b not in set(table.tolist())]
    untouched = kp.view(torch.int16)[:, spare] if layout == "per_layer" else kp.view(torch.int16)[spare]
    assert (untouched == 0x1357).all()
    S.close()


@pytest.mark.parametrize("seed", range(8))
def test_random_grouped_calls_match_separate_calls(ctx, seed):
    # deliveries spread over several sets in one cm_ingest_many, then one cm_render_many:
    # every set's ids, order and bytes equal its own cm_ingest_batch + cm_render
    rng = np.random.default_rng(4000 + seed)
    frags, _, _ = _case(200 + seed)
    L, H, _, d = frags[0][0].shape
    n_sets = int(rng.integers(1, 5))
    plan = [(int(rng.integers(0, n_sets)), int(rng.integers(0, len(frags))))
            for _ in range(int(rng.integers(1, 9)))]
    sets = [cm.FragmentSet(ctx) for _ in range(n_sets)]
    res = cm.ingest_many([(sets[s], *frags[f]) for s, f in plan])
    outs = [empty_out(L, H, max(S.seq_len(), 1) + int(rng.integers(0, 9)), d) for S in sets]
    lens = cm.render_many([(S, k, v) for S, (k, v) in zip(sets, outs)])
    torch.cuda.synchronize()
    for si, S in enumerate(sets):
        mine = [f for s, f in plan if s == si]
        T = cm.FragmentSet(ctx)
        ref = T.ingest_batch([frags[f] for f in mine])
        assert [r for (s, _), r in zip(plan, res) if s == si] == ref
        k, v = empty_out(L, H, max(T.seq_len(), 1), d)
        n, _ = T.render(k, v)
        torch.cuda.synchronize()
        assert lens[si] == n
        assert torch.equal(outs[si][0][:, :, :n], k[:, :, :n]) and torch.equal(outs[si][1][:, :, :n], v[:, :, :n])
        T.close()
    for S in sets:
        S.close()


@pytest.mark.parametrize("seed", range(8))
def test_random_incremental_render_matches_full_render(ctx, seed):
    # fragments arrive in two waves; the second render reuses the first's canonical prefix
    rng = np.random.default_rng(5000 + seed)
    frags, _, _ = _case(300 + seed)
    L, H, _, d = frags[0][0].shape
    cut = int(rng.integers(0, len(frags) + 1))
    total = sum(K.shape[2] for K, _ in frags)
    S = cm.FragmentSet(ctx)
    k, v = empty_out(L, H, total, d)
    S.ingest_batch(frags[:cut])
    _, order = S.render(k, v) if cut else (0, [])
    S.ingest_batch(frags[cut:])
    n, order2, reused = S.render_incremental(k, v, order)
    torch.cuda.synchronize()
    T = cm.FragmentSet(ctx)
    T.ingest_batch(frags)
    kf, vf = empty_out(L, H, total, d)
    nf, orderf = T.render(kf, vf)
    torch.cuda.synchronize()
    assert n == nf == total and order2 == orderf and 0 <= reused <= total
    assert torch.equal(k, kf) and torch.equal(v, vf)
    S.close()
    T.close()
