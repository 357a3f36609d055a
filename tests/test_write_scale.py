"""The write path's scale arithmetic, checked exhaustively on the CPU.

The GPU write computes fp32(amax) / 126.5 without a division: q0 = amax * y with
y = RN(1/126.5), then one correction with the remainder r = amax - q0 * 126.5
(exact in an FMA), q = RN(q0 + r * y) (Markstein's correction step).  amax is
the largest |x| of an fp16 row, so it is one of the 31744 finite non-negative
fp16 values; here every one of them is run through those steps with exact
rational arithmetic and a single round-to-nearest-even per FMA, and the result
must be the correctly rounded fp32 quotient, its fp16 rounding the oracle's
scale."""

import math
from fractions import Fraction

import numpy as np

from oracle import quantizer as OQ


def _rn32(x: Fraction) -> Fraction:
    """Nearest-even binary32 value of a non-negative rational (normal range)."""
    if x == 0:
        return Fraction(0)
    e = math.floor(math.log2(x.numerator) - math.log2(x.denominator))
    while Fraction(2) ** e > x:
        e -= 1
    while Fraction(2) ** (e + 1) <= x:
        e += 1
    ulp = Fraction(2) ** (max(e, -126) - 23)
    q, r = divmod(x, ulp)
    if 2 * r > ulp or (2 * r == ulp and q % 2 == 1):
        q += 1
    return q * ulp


def test_scale_division_equals_ieee_quotient_for_every_fp16_amax():
    b = Fraction(253, 2)                      # 126.5
    y = _rn32(1 / b)
    assert float(y) == float(np.float32(1.0) / np.float32(126.5))
    assert float(y) == float.fromhex("0x1.03091cp-7")
    amax = np.arange(0, 0x7C00, dtype=np.uint16).view(np.float16)   # 0 .. 65504
    got = np.empty(amax.size, dtype=np.float64)
    for i, a16 in enumerate(amax):
        a = Fraction(float(a16))
        q0 = _rn32(a * y)
        rem = a - q0 * b
        assert _rn32(abs(rem)) == abs(rem)    # the FMA remainder is exact
        q = _rn32(rem * y + q0) if rem >= 0 else _rn32(q0 - (-rem) * y)
        assert q == _rn32(a / b), float(a16)
        got[i] = float(q)
    ieee = amax.astype(np.float32) / np.float32(126.5)
    assert np.array_equal(got.astype(np.float32), ieee)
    # and the fp16 scale the write stores is the oracle's (rows whose amax is that value)
    s = got.astype(np.float32).astype(np.float16)
    s = np.where((s == 0) & (amax > 0), np.float16(2.0 ** -24), s)
    assert np.array_equal(s.view(np.uint16), OQ.scale_of_amax(amax.astype(np.float64)).view(np.uint16))


def test_rn32_helper_against_numpy():
    # the rounding helper itself, on a spread of rationals, against float32 casts of exact float64 values
    r = np.random.default_rng(0)
    for _ in range(2000):
        x = float(r.uniform(1e-6, 1e6))
        assert float(_rn32(Fraction(x))) == float(np.float32(x))
