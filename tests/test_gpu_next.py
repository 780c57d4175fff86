"""GPU tests of the rows after the hot path proper: incremental render (the lazy
O(m) re-render of Section 7) and render into a paged, block-table KV cache
(Section 4.5). Both must give the same bytes as a full contiguous render, which
the other suites tie to the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


@pytest.fixture(scope="module")
def ctx():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    c = cm.Context(0, THETA)
    yield c
    c.close()


def _frag(L, H, T, d, scale, seed):
    g = torch.Generator(device="cuda:0").manual_seed(seed)
    K = (torch.randn((L, H, T, d), generator=g, device="cuda:0") * scale).to(torch.bfloat16)
    V = torch.randn((L, H, T, d), generator=g, device="cuda:0").to(torch.bfloat16)
    return K, V


def _full_render(ctx, frags, cap):
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    L, H, _, d = frags[0][0].shape
    k, v = empty_out(L, H, cap, d, fill=0x1234)
    n, order = S.render(k, v)
    torch.cuda.synchronize()
    S.close()
    return k, v, order


def test_incremental_render_reuses_the_common_prefix(ctx):
    L, H, d = 4, 2, 128
    # scales set the canonical order: larger K norm renders earlier
    A = _frag(L, H, 300, d, 2.0, 1)
    B = _frag(L, H, 200, d, 1.0, 2)
    late = _frag(L, H, 150, d, 0.5, 3)     # sorts after A and B
    first = _frag(L, H, 100, d, 4.0, 4)    # sorts before everything
    mid = _frag(L, H, 120, d, 1.5, 5)      # sorts between A and B
    cap = 300 + 200 + 150 + 100 + 120
    S = cm.FragmentSet(ctx)
    S.ingest_batch([A, B])
    k, v = empty_out(L, H, cap, d, fill=0x1234)
    n, order = S.render(k, v)
    steps = [(late, 500), (first, 0), (mid, 100 + 300)]
    have = [A, B]
    for frag, reused_want in steps:
        S.ingest(*frag)
        have.append(frag)
        n, order, reused = S.render_incremental(k, v, order)
        torch.cuda.synchronize()
        assert reused == reused_want
        kf, vf, order_full = _full_render(ctx, have, cap)
        assert order == order_full
        assert torch.equal(k[:, :, :n], kf[:, :, :n]) and torch.equal(v[:, :, :n], vf[:, :, :n])
    # a stale or unrelated previous order falls back to a full render
    n, order2, reused = S.render_incremental(k, v, [bytes(16)] * 3)
    assert reused == 0 and order2 == order
    ref = oracle.from_deliveries([oracle_fragment(K, V) for K, V in have])
    K_ref, V_ref, o_order = oracle.render(ref, THETA)
    torch.cuda.synchronize()
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v[:, :, :n]), V_ref)
    assert assert_k_parity(synthetic.to_bits(k[:, :, :n]), K_ref) == 0
    S.close()


def _paged_check(ctx, frags, block_size, layout, seed):
    L, H, _, d = frags[0][0].shape
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    total = S.seq_len()
    nb_used = -(-total // block_size)
    num_blocks = nb_used + 7
    rng = np.random.default_rng(seed)
    table = torch.from_numpy(rng.permutation(num_blocks)[:nb_used].astype(np.int32)).to("cuda:0")
    if layout == "per_layer":          # [L][num_blocks][block_size][H][d]
        shape = (L, num_blocks, block_size, H, d)
        strides = dict(stride_layer=num_blocks * block_size * H * d, stride_block=block_size * H * d,
                       stride_token=H * d, stride_head=d)
    else:                              # [num_blocks][L][H][block_size][d]
        shape = (num_blocks, L, H, block_size, d)
        strides = dict(stride_block=L * H * block_size * d, stride_layer=H * block_size * d,
                       stride_head=block_size * d, stride_token=d)
    kp = torch.full(shape, 0, dtype=torch.int16, device="cuda:0").fill_(0x2468).view(torch.bfloat16)
    vp = torch.full(shape, 0, dtype=torch.int16, device="cuda:0").fill_(0x2468).view(torch.bfloat16)
    cache = cm.cm_paged_cache(kp.data_ptr(), vp.data_ptr(), table.data_ptr(), nb_used, block_size,
                              **strides)
    n, order = cm.cm_render_paged(S.handle, cache)
    torch.cuda.synchronize()
    kc, vc, order_c = _full_render(ctx, frags, total)
    assert n == total and order == order_c
    # gather the paged result back into [L][H][T][d]
    pos = torch.arange(total, device="cuda:0")
    blk = table.long()[pos // block_size]
    off = pos % block_size
    if layout == "per_layer":
        kg = kp[:, blk, off].permute(0, 2, 1, 3)
        vg = vp[:, blk, off].permute(0, 2, 1, 3)
    else:
        kg = kp[blk, :, :, off].permute(1, 2, 0, 3)
        vg = vp[blk, :, :, off].permute(1, 2, 0, 3)
    assert torch.equal(kg, kc) and torch.equal(vg, vc)
    # and the gathered paged result against the oracle directly
    K_ref, V_ref, o_order = oracle.render(
        oracle.from_deliveries([oracle_fragment(K, V) for K, V in frags]), THETA)
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(vg), V_ref)
    assert assert_k_parity(synthetic.to_bits(kg), K_ref) == 0
    # the spare blocks and the tail of the last used block are untouched
    used = set(table.tolist())
    spare = [b for b in range(num_blocks) if b not in used]
    if layout == "per_layer":
        untouched = kp.view(torch.int16)[:, spare]
    else:
        untouched = kp.view(torch.int16)[spare]
    assert (untouched == 0x2468).all()
    S.close()


# block sizes: powers of two no smaller than an item's rows (one table lookup per block an
# item touches: 16 at d = 128, 32 at d = 64 where the rows equal the block, 128 at d = 256)
# and the per-row lookups otherwise (12: not a power of two; 1 and 64 at d = 16: an item
# of 128 rows spans several blocks)
@pytest.mark.parametrize("layout,block_size,d", [("per_layer", 16, 128), ("block_major", 12, 64),
                                                 ("per_layer", 1, 16), ("block_major", 128, 256),
                                                 ("per_layer", 32, 64), ("block_major", 64, 16)])
def test_paged_render_matches_contiguous_render(ctx, layout, block_size, d):
    L, H = 3, 2
    frags = [_frag(L, H, T, d, 0.5 + 0.4 * i, 10 + i) for i, T in enumerate([37, 200, 5, 129])]
    _paged_check(ctx, frags, block_size, layout, seed=block_size)


def test_paged_render_q4b_shape(ctx):
    w = synthetic.WORKLOADS["q4b_t512"]
    specs = synthetic.fragment_specs(w)
    frags = [synthetic.make_fragment_torch(sp, w.num_layers, w.num_kv_heads, w.head_dim, "cuda:0")
             for sp in specs]
    _paged_check(ctx, frags, 16, "per_layer", seed=3)


def test_paged_render_rejects_bad_descriptors(ctx):
    K, V = _frag(2, 1, 20, 64, 1.0, 7)
    S = cm.FragmentSet(ctx)
    S.ingest(K, V)
    pool = torch.empty((2, 4, 16, 1, 64), dtype=torch.bfloat16, device="cuda:0")
    table = torch.arange(4, dtype=torch.int32, device="cuda:0")
    ok = dict(stride_layer=4 * 16 * 64, stride_block=16 * 64, stride_token=64, stride_head=64)
    short = cm.cm_paged_cache(pool.data_ptr(), pool.data_ptr(), table.data_ptr(), 1, 16, **ok)
    with pytest.raises(cm.CMError) as e:
        cm.cm_render_paged(S.handle, short)
    assert e.value.status == cm.Status.ERR_CAPACITY
    bad = dict(ok, stride_token=60)
    odd = cm.cm_paged_cache(pool.data_ptr(), pool.data_ptr(), table.data_ptr(), 4, 16, **bad)
    with pytest.raises(cm.CMError) as e:
        cm.cm_render_paged(S.handle, odd)
    assert e.value.status == cm.Status.ERR_ALIGNMENT
    S.close()
