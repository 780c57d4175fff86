"""Mean K-norm score rho_i and its integer key (test infrastructure only).

Eq. rho (Section 4.3) and Algorithm 1: at the routing layer l*, rho_i is the
mean over batch, heads and the last T* = min_j T_j positions of the L2 norm of
K_i^{(l*)}[b, h, t, :]. Readings:
  * the norm is taken per (head, position) over head_dim, then averaged
    ("averaged over batch and heads"), not one Frobenius norm over heads x d;
  * l* is 0-indexed here, default floor(L/2) (the paper's 1-indexed l* = 15 for
    28 layers is the same layer as 0-indexed 14);
  * to make the order exact and independent of any summation order, the score
    is carried as an integer: per row the squared norm is summed in fp64 over
    head_dim in ascending element order, n = sqrt(ss) (correctly rounded),
    q = round-half-even(n * 2^20) saturated at 2^44 - 1 (NaN and inf saturate),
    and Q[t] = sum over heads of q(h, t). The tail sum S_i of Q over the last
    T* positions equals rho_i * H * T* * 2^20 up to the quantisation, so the
    order by S is the order by rho wherever their gaps exceed 2^-20.
"""
from __future__ import annotations

import numpy as np

from .bf16 import bits_to_f64

NORM_SCALE_EXP = 20
Q_MAX = (1 << 44) - 1


def default_routing_layer(L: int) -> int:
    return L // 2


def row_norms_fp64(K_layer_bits: np.ndarray) -> np.ndarray:
    """n(h, t) = sqrt(sum_e x_e^2), the sum taken in fp64 in ascending e order.

    K_layer_bits is [H, T, d] uint16. Each x^2 of a bf16 value is exact in fp64.
    """
    x = bits_to_f64(K_layer_bits)
    ss = np.zeros(x.shape[:-1], dtype=np.float64)
    for e in range(x.shape[-1]):        # sequential, ascending e (no pairwise sum)
        ss = ss + x[..., e] * x[..., e]
    return np.sqrt(ss)


def quantise(n: np.ndarray) -> np.ndarray:
    """q = round-half-even(n * 2^20), saturated at 2^44 - 1; NaN/inf saturate."""
    with np.errstate(invalid="ignore", over="ignore"):
        scaled = np.ldexp(n, NORM_SCALE_EXP)
        sat = ~np.isfinite(scaled) | (scaled >= float(Q_MAX))
        r = np.rint(np.where(sat, 0.0, scaled))
    q = r.astype(np.uint64)
    return np.where(sat, np.uint64(Q_MAX), q).astype(np.uint64)


def norm_key(K_bits: np.ndarray, routing_layer: int) -> np.ndarray:
    """Q[t] = sum_h q(h, t) at the routing layer, uint64 of length T."""
    q = quantise(row_norms_fp64(K_bits[routing_layer]))     # [H, T]
    Q = np.zeros(q.shape[1], dtype=np.uint64)
    for h in range(q.shape[0]):
        Q = Q + q[h]
    return Q


def tail_sum(Q: np.ndarray, t_star: int) -> int:
    """S_i = sum of Q over the last T* positions (0-based [T-T*, T)), exact."""
    T = Q.shape[0]
    return sum(int(v) for v in Q[T - t_star:T])


def rho_fp64(K_bits: np.ndarray, routing_layer: int, t_star: int) -> float:
    """rho_i of Eq. rho in fp64, without quantisation (cross-check only)."""
    n = row_norms_fp64(K_bits[routing_layer])          # [H, T]
    T = n.shape[1]
    return float(np.mean(n[:, T - t_star:T]))
