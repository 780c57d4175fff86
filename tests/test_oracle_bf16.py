"""Pins for the oracle's bf16 conversions (CPU only).

The decode is pinned to known bit patterns; the encode to torch's binary32 ->
bf16 conversion (round half to even) on binary32-representable inputs, and to
an exact rational nearest-value search on fp64 inputs that binary32 cannot hold.
"""
import bisect
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle.bf16 import bits_to_f64, f64_to_bits, ulp_distance, is_nan_bits


def test_decode_known_patterns():
    bits = np.array([0x3F80, 0xC000, 0x0001, 0x0080, 0x7F7F, 0x7F80, 0xFF80, 0x8000, 0x3FC0],
                    dtype=np.uint16)
    want = [1.0, -2.0, 2.0 ** -133, 2.0 ** -126, (2 - 2 ** -7) * 2.0 ** 127,
            np.inf, -np.inf, -0.0, 1.5]
    got = bits_to_f64(bits)
    assert list(got) == want
    assert np.signbit(got[7])


def _torch_bits(x32: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(x32).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def test_encode_matches_torch_on_binary32_inputs():
    rng = np.random.default_rng(7)
    raw = rng.integers(0, 2 ** 32, size=200_000, dtype=np.uint64).astype(np.uint32)
    # force exact ties, near-ties, subnormals and values near the top of the range
    raw[:2000] = (raw[:2000] & np.uint32(0xFFFF0000)) | np.uint32(0x8000)
    raw[2000:4000] = (raw[2000:4000] & np.uint32(0xFFFF0000)) | np.uint32(0x7FFF)
    raw[4000:6000] = raw[4000:6000] & np.uint32(0x807FFFFF)          # subnormal binary32
    raw[6000:8000] = (raw[6000:8000] & np.uint32(0x8000FFFF)) | np.uint32(0x7F7F0000)
    x32 = raw.view(np.float32)
    keep = ~np.isnan(x32)
    x32 = x32[keep]
    ours = f64_to_bits(x32.astype(np.float64))
    theirs = _torch_bits(x32)
    assert np.array_equal(ours, theirs)


def _all_positive_finite_bf16():
    bits = np.arange(0, 0x7F80, dtype=np.uint16)
    return [Fraction(float(v)) for v in bits_to_f64(bits)], bits


def _exact_nearest_bits(x: float, table, table_bits) -> int:
    """Nearest bf16 by exact rational comparison, ties to even; +-inf past the top."""
    if x != x:
        return 0x7FC0
    sign = 0x8000 if (x < 0 or (x == 0 and np.signbit(x))) else 0
    a = abs(Fraction(x))
    top = table[-1]
    half_top_ulp = Fraction(2) ** 119      # half the spacing just below 2^128
    if a >= top + half_top_ulp:
        return sign | 0x7F80
    i = bisect.bisect_left(table, a)
    if i < len(table) and table[i] == a:
        return sign | int(table_bits[i])
    lo, hi = i - 1, i
    if hi == len(table):                      # between the top value and the overflow point
        return sign | int(table_bits[lo])
    dlo, dhi = a - table[lo], table[hi] - a
    if dlo < dhi:
        pick = lo
    elif dhi < dlo:
        pick = hi
    else:
        pick = lo if (int(table_bits[lo]) & 1) == 0 else hi
    return sign | int(table_bits[pick])


def test_encode_matches_exact_rational_rounding_on_fp64_inputs():
    table, table_bits = _all_positive_finite_bf16()
    rng = np.random.default_rng(11)
    xs = list(rng.standard_normal(3000) * np.exp(rng.uniform(-90, 88, 3000)))
    # values a hair off bf16 midpoints (not binary32 values): double rounding would fail here
    for b in rng.integers(0x0080, 0x7F00, 500):
        mid = (float(bits_to_f64(np.uint16(b))) + float(bits_to_f64(np.uint16(b + 1)))) / 2
        xs += [mid, np.nextafter(mid, np.inf), np.nextafter(mid, -np.inf), -mid]
    # subnormal range, overflow edge, signed zeros
    xs += list(rng.uniform(-2.0 ** -126, 2.0 ** -126, 500))
    top = (2 - 2 ** -7) * 2.0 ** 127
    xs += [top, top * (1 + 2 ** -9), top * (1 + 2 ** -8), 2.0 ** 128 * (1 - 2 ** -9), 1e39,
           -1e39, 0.0, -0.0, 2.0 ** -134, 2.0 ** -134 * 1.0000001, 3 * 2.0 ** -134]
    x = np.array(xs, dtype=np.float64)
    got = f64_to_bits(x)
    want = np.array([_exact_nearest_bits(v, table, table_bits) for v in xs], dtype=np.uint16)
    assert np.array_equal(got, want)


def test_nan_and_signed_zero():
    got = f64_to_bits(np.array([np.nan, -0.0, 0.0]))
    assert is_nan_bits(got[:1]).all()
    assert got[1] == 0x8000 and got[2] == 0x0000


@pytest.mark.parametrize("a,b,dist", [(0x0000, 0x8000, 0), (0x3F80, 0x3F81, 1),
                                      (0x0001, 0x8001, 2), (0x7F7F, 0x7F80, 1)])
def test_ulp_distance(a, b, dist):
    assert ulp_distance(np.uint16(a), np.uint16(b)) == dist
