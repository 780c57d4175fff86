"""Canonical order and render (test infrastructure only).

CanonicalMerge (Algorithm 1, Section 4.3): order the fragments by descending
mean K-norm rho at the routing layer, ties broken by descending content hash,
then apply BagMerge (Section 4.2, Eq. bagmerge-k / bagmerge-v) in that order.
Render(S) (Algorithm 2) is CanonicalMerge over the fragments of the set.

BagMerge with order pi: offsets s_pi(1) = 0, s_pi(i) = s_pi(i-1) + T_pi(i-1);
for every layer, K* is the sequence-axis concatenation of R(s) R(0)^-1 K_pi(i)
and V* that of V_pi(i). K is stored post-rotation, R(t) k at position t, and
R(0) is the identity, so each stored key becomes R(s) R(t) k = R(s + t) k: one
rotation by the slot's constant offset s (the delta formula of Section 2.3).

Readings:
  * RoPE pairing: rotate-half, element j pairs with j + d/2, frequency
    w_j = theta^(-2j/d); (x, y) -> (x cos a - y sin a, y cos a + x sin a),
    a = s * w_j. Angles, cos and sin are fp64 (the host math library); the two
    products and the sum are fp64, then one direct round to bf16.
  * The slot at offset 0 keeps its original rotation, so its K is copied as
    bytes (arithmetic with cos = 1, sin = 0 could flip the sign of a zero).
  * V is copied as bytes.
  * The tie-break compares the 16-byte id as a big-endian integer, descending.
  * T* is the minimum length over the fragments of the set; the empty set
    renders to length 0.
"""
from __future__ import annotations

import math
from typing import List, Sequence, Tuple

import numpy as np

from .bf16 import bits_to_f64, f64_to_bits
from .content_address import id_as_int
from .fragment_set import Fragment, FragmentSet
from .norm import tail_sum


def canonical_order(fragments: Sequence[Fragment]) -> Tuple[List[Fragment], List[int]]:
    """pi* = argsort_i(-rho_i, -h_i) with rho carried as the integer tail sum S_i."""
    if not fragments:
        return [], []
    t_star = min(f.seq_len for f in fragments)
    keyed = [(tail_sum(f.Q, t_star), id_as_int(f.fid), f) for f in fragments]
    keyed.sort(key=lambda k: (-k[0], -k[1]))
    return [k[2] for k in keyed], [k[0] for k in keyed]


def offsets(order: Sequence[Fragment]) -> List[int]:
    """s_pi(1) = 0, s_pi(i) = s_pi(i-1) + T_pi(i-1)."""
    out, s = [], 0
    for f in order:
        out.append(s)
        s += f.seq_len
    return out


def delta_cos_sin(s: int, d: int, theta: float):
    """fp64 cos and sin of a_j = s * theta^(-2j/d), j < d/2."""
    c = np.empty(d // 2, dtype=np.float64)
    sn = np.empty(d // 2, dtype=np.float64)
    for j in range(d // 2):
        w = theta ** (-(2.0 * j) / d)
        a = float(s) * w
        c[j] = math.cos(a)
        sn[j] = math.sin(a)
    return c, sn


def rotate_pairs_f64(x: np.ndarray, y: np.ndarray, s: int, theta: float):
    """R(s) on fp64 halves x = k[..., :d/2], y = k[..., d/2:], without rounding."""
    d = 2 * x.shape[-1]
    c, sn = delta_cos_sin(s, d, theta)
    xr = x * c - y * sn          # two fp64 products, one fp64 difference
    yr = y * c + x * sn
    return xr, yr


def rotate_k(K_bits: np.ndarray, s: int, theta: float) -> np.ndarray:
    """R(s) applied to stored keys [..., d]; s = 0 is a byte copy."""
    if s == 0:
        return K_bits.copy()
    half = K_bits.shape[-1] // 2
    xr, yr = rotate_pairs_f64(bits_to_f64(K_bits[..., :half]),
                              bits_to_f64(K_bits[..., half:]), s, theta)
    out = np.empty_like(K_bits)
    out[..., :half] = f64_to_bits(xr)
    out[..., half:] = f64_to_bits(yr)
    return out


def bagmerge(order: Sequence[Fragment], theta: float) -> Tuple[np.ndarray, np.ndarray]:
    """BagMerge(pi) for fragments already listed in order pi: (K*, V*) uint16 [L, H, sum T, d]."""
    if not order:
        return np.zeros((0, 0, 0, 0), np.uint16), np.zeros((0, 0, 0, 0), np.uint16)
    L, H, _, d = order[0].shape
    total = sum(f.seq_len for f in order)
    K_out = np.empty((L, H, total, d), dtype=np.uint16)
    V_out = np.empty((L, H, total, d), dtype=np.uint16)
    for f, s in zip(order, offsets(order)):
        T = f.seq_len
        K_out[:, :, s:s + T, :] = rotate_k(f.K, s, theta)
        V_out[:, :, s:s + T, :] = f.V
    return K_out, V_out


def canonical_merge(fragments: Sequence[Fragment], theta: float):
    """Algorithm 1: (K*, V*, canonical order)."""
    order, _ = canonical_order(fragments)
    K, V = bagmerge(order, theta)
    return K, V, order


def render(S: FragmentSet, theta: float):
    """Algorithm 2, Render(S): CanonicalMerge over the fragments of the set."""
    return canonical_merge(S.fragments(), theta)


def naive_multiset_render(deliveries: Sequence[Fragment], theta: float):
    """Section 5.9 foil: every delivery is a fresh operand, duplicates included."""
    return canonical_merge(list(deliveries), theta)
