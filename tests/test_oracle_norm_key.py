"""Pins for the oracle's norm key (Eq. rho) (CPU only): closed forms, tail
alignment, agreement of the integer key with the fp64 score, saturation."""
import math

import numpy as np
import pytest

from oracle.bf16 import bits_to_f64, f64_to_bits
import oracle.norm as nk
from oracle.merge import rotate_k
from synthetic import random_bits


def _const_layer(values_ht, d):
    """[H, T, d] bits whose row (h, t) is values_ht[h][t] repeated d times."""
    v = np.asarray(values_ht, dtype=np.float64)
    return np.repeat(f64_to_bits(v)[..., None], d, axis=-1)


@pytest.mark.parametrize("d,root", [(16, 4), (64, 8), (256, 16)])
def test_constant_rows_closed_form(d, root):
    # a row of d equal entries x has norm |x| sqrt(d); for d a power of 4 this is exact
    xs = bits_to_f64(f64_to_bits(np.array([[0.75, -1.5, 3.0], [2.0 ** -10, 7.0, -0.0]])))
    K = np.zeros((3, 2, 3, d), dtype=np.uint16)
    K[1] = _const_layer(xs, d)
    Q = nk.norm_key(K, 1)
    q = np.rint(np.abs(xs) * root * 2.0 ** 20).astype(np.uint64)
    assert list(Q) == [int(q[0, t] + q[1, t]) for t in range(3)]


def test_pythagorean_rows():
    # (3a, 4a, 0, ...) has norm 5a exactly
    d = 128
    K = np.zeros((1, 1, 4, d), dtype=np.uint16)
    for t, a in enumerate([1.0, 0.5, 2.0 ** -20, 96.0]):
        K[0, 0, t, 7] = f64_to_bits(np.float64(3 * a))
        K[0, 0, t, 100] = f64_to_bits(np.float64(-4 * a))
    Q = nk.norm_key(K, 0)
    assert list(Q) == [int(round(5 * a * 2 ** 20)) for a in [1.0, 0.5, 2.0 ** -20, 96.0]]


def test_tail_alignment_uses_last_t_star_positions():
    # fragment A: large norms at its head, small at its tail; B: uniform medium norms.
    d = 16
    A = np.zeros((1, 1, 10, d), dtype=np.uint16)
    A[0] = _const_layer([[8.0] * 6 + [0.5] * 4], d)
    B = np.zeros((1, 1, 4, d), dtype=np.uint16)
    B[0] = _const_layer([[1.0] * 4], d)
    QA, QB = nk.norm_key(A, 0), nk.norm_key(B, 0)
    t_star = 4
    # tail of A is four rows of 0.5 * sqrt(16) = 2; B is four rows of 4
    assert nk.tail_sum(QA, t_star) == 4 * 2 * 2 ** 20
    assert nk.tail_sum(QB, t_star) == 4 * 4 * 2 ** 20
    # whole-length means would rank A first; the tail-aligned key ranks B first
    assert QA.astype(np.float64).mean() > QB.astype(np.float64).mean()
    assert nk.tail_sum(QB, t_star) > nk.tail_sum(QA, t_star)


def test_integer_key_agrees_with_fp64_rho():
    rng = np.random.default_rng(1)
    for T in (5, 37, 200):
        K = random_bits(rng, (4, 3, T, 64), scale=float(rng.uniform(0.5, 1.5)))
        Q = nk.norm_key(K, 2)
        for t_star in (1, T // 2 + 1, T):
            rho_from_key = nk.tail_sum(Q, t_star) / (2.0 ** 20 * 3 * t_star)
            assert abs(rho_from_key - nk.rho_fp64(K, 2, t_star)) <= 2.0 ** -21


def test_rotation_preserves_norm_within_bf16_rounding():
    rng = np.random.default_rng(2)
    K = random_bits(rng, (1, 2, 50, 128))
    n0 = nk.row_norms_fp64(K[0])
    n1 = nk.row_norms_fp64(rotate_k(K, 1234, 1e6)[0])
    assert np.all(np.abs(n1 - n0) <= 2.0 ** -8 * n0)


def test_saturation_and_nonfinite():
    d = 16
    K = np.zeros((1, 1, 3, d), dtype=np.uint16)
    K[0, 0, 0, :] = 0x7F7F           # largest finite bf16: norm ~1.36e39, saturates
    K[0, 0, 1, 0] = 0x7FC0           # NaN
    K[0, 0, 2, 0] = 0x7F80           # inf
    assert list(nk.norm_key(K, 0)) == [nk.Q_MAX] * 3


def test_sum_over_heads_and_default_layer():
    assert nk.default_routing_layer(28) == 14 and nk.default_routing_layer(36) == 18
    rng = np.random.default_rng(4)
    K = random_bits(rng, (3, 5, 7, 32))
    n = nk.row_norms_fp64(K[1])
    q = [[int(round(float(v) * 2 ** 20)) if abs(v * 2 ** 20 - math.floor(v * 2 ** 20) - 0.5) > 1e-9
          else None for v in row] for row in n]
    Q = nk.norm_key(K, 1)
    for t in range(7):
        if all(q[h][t] is not None for h in range(5)):
            assert int(Q[t]) == sum(q[h][t] for h in range(5))


# rows of d = 16 equal entries k 2^-23 have norm 4 k 2^-23, so 2^20 n = k / 2 exactly:
# half-integers for odd k, which round half to even (0.5 -> 0, 1.5 -> 2, 2.5 -> 2,
# 3.5 -> 4, 4.5 -> 4); floor(x + 0.5) or rounding half away from zero would give
# 1, 2, 3, 4, 5
HALF_TIE_K = [1, 3, 5, 7, 9]
HALF_TIE_Q = [0, 2, 2, 4, 4]


def test_quantise_rounds_exact_halves_to_even():
    n = np.array([k * 2.0 ** -21 for k in HALF_TIE_K])          # 2^20 n = k / 2
    assert list(nk.quantise(n)) == HALF_TIE_Q
    K = np.zeros((2, 1, len(HALF_TIE_K), 16), dtype=np.uint16)
    K[1] = _const_layer([[k * 2.0 ** -23 for k in HALF_TIE_K]], 16)
    assert list(nk.norm_key(K, 1)) == HALF_TIE_Q
    # two heads: each adds its own rounded term
    K2 = np.zeros((2, 2, len(HALF_TIE_K), 16), dtype=np.uint16)
    K2[1] = _const_layer([[k * 2.0 ** -23 for k in HALF_TIE_K]] * 2, 16)
    assert list(nk.norm_key(K2, 1)) == [2 * q for q in HALF_TIE_Q]
