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
