"""Exact binary32 arithmetic for the tests, independent of any float unit.

``round_f32(q)`` rounds an exact rational to the nearest binary32 value, ties to
even, with subnormals (IEEE 754-2019, Sec. 4.3.1). The tests use it to state what
a correctly rounded fused multiply-add must return, without calling fmaf.
"""
from fractions import Fraction
import math
import struct

import numpy as np

_EMIN = -126          # smallest normal exponent of binary32
_P = 24               # precision in bits
_MAX = Fraction((2 ** 24 - 1) * 2 ** 104)   # largest finite binary32


def to_frac(x) -> Fraction:
    x = float(x)
    if not math.isfinite(x):
        raise ValueError("not finite")
    return Fraction(x)


def _floor_log2(q: Fraction) -> int:
    n, d = q.numerator, q.denominator
    e = n.bit_length() - d.bit_length()
    # adjust so that 2**e <= q < 2**(e+1)
    if e >= 0:
        if n < (d << e):
            e -= 1
    else:
        if (n << -e) < d:
            e -= 1
    return e


def round_f32(q: Fraction) -> float:
    """Round an exact rational to binary32 (RNE). Zero returns +0.0."""
    if q == 0:
        return 0.0
    sign = -1.0 if q < 0 else 1.0
    m = abs(q)
    e = max(_floor_log2(m), _EMIN)
    ulp = Fraction(2) ** (e - (_P - 1))
    r = m / ulp
    fl = r.numerator // r.denominator
    rem = r - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    val = fl * ulp
    if val > _MAX:
        return sign * math.inf
    out = sign * float(val)
    assert np.float32(out) == out  # representable by construction
    return out


def fma_f32(a, b, c) -> float:
    """Correctly rounded binary32 a*b + c for finite binary32 inputs."""
    return round_f32(to_frac(a) * to_frac(b) + to_frac(c))


def f32_bits(x) -> int:
    return struct.unpack("<I", struct.pack("<f", float(x)))[0]


def ulp_f32(x) -> Fraction:
    """Spacing of binary32 numbers at |x| (the subnormal spacing near zero)."""
    m = abs(to_frac(x))
    if m == 0:
        return Fraction(2) ** (_EMIN - (_P - 1))
    e = max(_floor_log2(m), _EMIN)
    return Fraction(2) ** (e - (_P - 1))
