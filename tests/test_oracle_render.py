"""Pins for the oracle's render (Eq. bagmerge-k/v, Algorithms 1 and 2) (CPU only):
offset-0 identity, rotation composition, agreement with complex multiplication
and with RoPE applied at the shifted positions, permutation invariance for
N <= 5, the paper's Appendix A lengths and Section 5.9 re-delivery lengths, and
the non-idempotence of the rendered operator (Section 4.4)."""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle.bf16 import bits_to_f64, f64_to_bits, ulp_distance
from synthetic import random_bits

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
THETA = 1.0e6


def test_offset_zero_is_a_byte_copy_including_signed_zeros():
    rng = np.random.default_rng(0)
    K = random_bits(rng, (2, 2, 5, 64))
    K[0, 0, 0, :4] = [0x8000, 0x0000, 0x8000, 0x0001]
    out = oracle.rotate_k(K, 0, THETA)
    assert np.array_equal(out, K)


@pytest.mark.parametrize("d", [8, 64, 128])
def test_rotation_composition_in_fp64(d):
    rng = np.random.default_rng(d)
    x = rng.standard_normal((5, d // 2))
    y = rng.standard_normal((5, d // 2))
    for a, b in [(1, 1), (3, 17), (512, 4096), (12345, 54321)]:
        x1, y1 = oracle.rotate_pairs_f64(x, y, a, THETA)
        x2, y2 = oracle.rotate_pairs_f64(x1, y1, b, THETA)
        x3, y3 = oracle.rotate_pairs_f64(x, y, a + b, THETA)
        scale = np.sqrt(x ** 2 + y ** 2)
        assert np.all(np.abs(x2 - x3) <= 1e-12 * (1 + scale) * (a + b) ** 0.5)
        assert np.all(np.abs(y2 - y3) <= 1e-12 * (1 + scale) * (a + b) ** 0.5)


def test_rotation_equals_complex_multiplication():
    # pair (x_j, y_j) as x_j + i y_j, rotated by a_j = s * theta^(-2j/d): multiply by e^{i a_j}
    d = 64
    rng = np.random.default_rng(1)
    x = rng.standard_normal((3, d // 2))
    y = rng.standard_normal((3, d // 2))
    for s in (1, 7, 300, 9999):
        a = s * np.power(THETA, -np.arange(0, d, 2) / d)
        z = (x + 1j * y) * np.exp(1j * a)
        xr, yr = oracle.rotate_pairs_f64(x, y, s, THETA)
        assert np.allclose(xr, z.real, rtol=0, atol=1e-12)
        assert np.allclose(yr, z.imag, rtol=0, atol=1e-12)


def test_unit_vectors_map_to_cos_sin():
    d = 16
    for j in range(d // 2):
        x = np.zeros((1, d // 2)); y = np.zeros((1, d // 2)); x[0, j] = 1.0
        xr, yr = oracle.rotate_pairs_f64(x, y, 5, THETA)
        a = 5 * THETA ** (-2.0 * j / d)
        assert xr[0, j] == pytest.approx(math.cos(a), abs=1e-15)
        assert yr[0, j] == pytest.approx(math.sin(a), abs=1e-15)
        assert np.count_nonzero(xr) + np.count_nonzero(yr) <= 2


def test_shift_of_stored_keys_equals_rope_at_shifted_positions():
    # keys generated in fp64 as R(t) u and stored in bf16, then shifted by s, agree with
    # R(s + t) u up to the bf16 rounding of the stored pair (relative 2^-8 per component at
    # worst, carried through the rotation) plus the final rounding (2^-8 relative) of each
    # side. A wrong pairing, sign or frequency would miss by O(1).
    d, T = 128, 40
    rng = np.random.default_rng(2)
    u = rng.standard_normal((1, 1, T, d))
    t = np.arange(T)[:, None]

    def rope_at(pos):
        a = pos * np.power(THETA, -np.arange(0, d, 2) / d)[None, :]
        z = (u[..., :d // 2] + 1j * u[..., d // 2:]) * np.exp(1j * a)
        return np.concatenate([z.real, z.imag], axis=-1)

    stored = f64_to_bits(rope_at(t))
    sv = bits_to_f64(stored)
    pair_mag = np.abs(sv[..., :d // 2]) + np.abs(sv[..., d // 2:])
    pair_mag = np.concatenate([pair_mag, pair_mag], axis=-1)
    for s in (1, 37, 4096):
        shifted = bits_to_f64(oracle.rotate_k(stored, s, THETA))
        exact = rope_at(t + s)
        bound = 2.0 ** -8 * pair_mag + 2.0 ** -8 * np.abs(exact) + 1e-30
        assert np.all(np.abs(shifted - exact) <= bound)
        ulps = ulp_distance(oracle.rotate_k(stored, s, THETA), f64_to_bits(exact))
        assert (ulps <= 1).mean() > 0.9


def _frags(lengths, L=2, H=2, d=16, seed=0):
    rng = np.random.default_rng(seed)
    out = []
    for i, T in enumerate(lengths):
        K = random_bits(rng, (L, H, T, d), scale=0.5 + 0.3 * i)
        V = random_bits(rng, (L, H, T, d))
        out.append(oracle.make_fragment(K, V))
    return out


def test_permutation_invariance_and_app_a_lengths():
    g = json.load(open(os.path.join(GOLDEN, "app_a_canonical_concat.json")))
    p = g["positions_per_thinker"]
    total_concat, total_arity = 0, 0
    for n in (2, 3, 4, 5):
        frags = _frags([p] * n, seed=n)
        K0, V0, _ = oracle.canonical_merge(frags, THETA)
        if str(n) in g["rendered_length"]:
            assert K0.shape[2] == g["rendered_length"][str(n)]
        for perm in itertools.permutations(frags):
            K, V, _ = oracle.canonical_merge(list(perm), THETA)
            assert np.array_equal(K, K0) and np.array_equal(V, V0)
            total_arity += 1
            total_concat += n <= 4
    assert total_concat == g["concat_permutations_total"]
    assert total_arity == g["arity_permutations_total"]


def test_layout_v_copied_and_k_slots_rotated_by_offset():
    frags = _frags([5, 3, 4], seed=5)
    K, V, order = oracle.canonical_merge(frags, THETA)
    s = 0
    for f in order:
        T = f.seq_len
        assert np.array_equal(V[:, :, s:s + T], f.V)
        if s == 0:
            assert np.array_equal(K[:, :, :T], f.K)
        else:
            assert np.array_equal(K[:, :, s:s + T], oracle.rotate_k(f.K, s, THETA))
            assert not np.array_equal(K[:, :, s:s + T], f.K)
        s += T


def test_redelivery_lengths_match_table_redeliver():
    g = json.load(open(os.path.join(GOLDEN, "redelivery.json")))
    total = g["crdt_seq_len"][0]
    a, b = _frags([total // 2 - 4, total // 2 + 4], L=1, H=1, d=16, seed=7)
    for R, naive_len, crdt_len in zip(g["R"], g["naive_seq_len"], g["crdt_seq_len"]):
        deliveries = []
        for _ in range(R):
            deliveries += [oracle.make_fragment(a.K.copy(), a.V.copy()),
                           oracle.make_fragment(b.K.copy(), b.V.copy())]
        S = oracle.from_deliveries(deliveries)
        assert len(S) == g["crdt_set_size"]
        K, V, _ = oracle.render(S, THETA)
        assert K.shape[2] == crdt_len
        Kn, _, _ = oracle.naive_multiset_render(deliveries, THETA)
        assert Kn.shape[2] == naive_len
        K1, V1, _ = oracle.render(oracle.from_deliveries([a, b]), THETA)
        assert np.array_equal(K, K1) and np.array_equal(V, V1)


def test_rendered_operator_is_not_idempotent():
    # CM(CM(A, B), B) != CM(A, B): the copy of B inside the merge has been shifted
    a, b = _frags([6, 6], seed=8)
    K, V, _ = oracle.canonical_merge([a, b], THETA)
    merged = oracle.make_fragment(K, V)
    K2, V2, _ = oracle.canonical_merge([merged, b], THETA)
    assert K2.shape != K.shape or not np.array_equal(K2, K)
    # whereas the state absorbs: render(S u {B}) == render(S)
    S = oracle.from_deliveries([a, b])
    assert oracle.union(S, oracle.from_deliveries([b])) == S


def test_empty_set_renders_to_length_zero():
    K, V, order = oracle.render(oracle.FragmentSet(), THETA)
    assert K.size == 0 and V.size == 0 and order == []
