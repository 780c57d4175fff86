"""bf16 <-> fp64 for the oracle (test infrastructure only).

bf16 is IEEE binary32 with the low 16 significand bits dropped: 1 sign bit,
8 exponent bits (bias 127), 7 stored significand bits, so 8 significant bits
for normal numbers and a subnormal spacing of 2^-133.

Decoding is exact: the bits shifted left by 16 are the binary32 pattern.
Encoding rounds an fp64 value *directly* to the nearest bf16, ties to even,
with no intermediate binary32 (which would round twice). Subnormals are kept,
values that round past the largest finite bf16 become +-inf, signed zeros keep
their sign, and NaN becomes the quiet NaN 0x7FC0.
"""
from __future__ import annotations

import numpy as np

BF16_QNAN = np.uint16(0x7FC0)
_SUBNORMAL_QUANTUM_EXP = -133  # spacing of bf16 subnormals is 2^-133


def bits_to_f64(bits) -> np.ndarray:
    """uint16 bf16 bit patterns -> float64 values (exact)."""
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def f64_to_bits(x) -> np.ndarray:
    """float64 -> nearest bf16 (round half to even), as uint16 bit patterns."""
    x = np.asarray(x, dtype=np.float64)
    with np.errstate(over="ignore", invalid="ignore"):
        # x = m * 2^e with 0.5 <= |m| < 1; a normal bf16 at that binade has
        # quantum 2^(e-8); below the normal range the quantum stays 2^-133.
        _, e = np.frexp(x)
        q_exp = np.maximum(e.astype(np.int64) - 8, _SUBNORMAL_QUANTUM_EXP)
        # scaling by a power of two is exact; rint rounds half to even
        r = np.ldexp(np.rint(np.ldexp(x, -q_exp)), q_exp)
        # r is now a bf16 value (or 2^128, which becomes inf), so the binary32
        # conversion below is exact and its low 16 bits are zero
        r32 = r.astype(np.float32)
    out = (r32.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
    out = np.where(np.isnan(x), BF16_QNAN, out)
    return out.astype(np.uint16)


def ulp_distance(a_bits, b_bits) -> np.ndarray:
    """Distance in bf16 ulps between two bit arrays, on the monotone integer
    ordering of bf16 (so +0 and -0 are both at distance 0 from each other)."""
    def ordered(b):
        b = np.asarray(b, dtype=np.uint16).astype(np.int64)
        mag = b & 0x7FFF
        return np.where(b & 0x8000, -mag, mag)
    return np.abs(ordered(a_bits) - ordered(b_bits))


def is_nan_bits(bits) -> np.ndarray:
    b = np.asarray(bits, dtype=np.uint16)
    return ((b & 0x7F80) == 0x7F80) & ((b & 0x007F) != 0)
