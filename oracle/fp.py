"""Floating-point encodings used by the cache, written from their definitions.

Test infrastructure only (see ``oracle/__init__.py``).

* IEEE binary16 round-to-nearest-even: numpy's float64 -> float16 cast
  (a library primitive, pinned against exact rational rounding in
  ``tests/test_oracle_fp.py``).
* binary16 round toward +infinity: the witness is stored in fp16 and must
  not under-state the residual norm (§4.1, Eq. witness: "stored in fp16";
  rounding up keeps Thm. "Sound black-box logit bound" sound).
* OCP fp8 E4M3 ("e4m3fn": no infinities, one NaN pattern per sign, largest
  finite 448, exponent bias 7, subnormals m * 2^-9) with round-to-nearest-
  even and saturation of finite overflow to +-448 -- the "raw-cast fp8-e4m3
  black-box scheme" of the six-quantizer study (§4.1, Fig. f5) taken as a
  cast with no scale.
"""

import numpy as np

FP16_MIN_SUBNORMAL = 2.0 ** -24
E4M3_MAX = 448.0


def fp16_rn(x):
    """Round float64 values to the nearest binary16 (ties to even)."""
    return np.asarray(x, dtype=np.float64).astype(np.float16)


def fp16_ru(x):
    """Round non-negative float64 values up to binary16 (toward +inf)."""
    x = np.asarray(x, dtype=np.float64)
    if np.any(x < 0) or np.any(np.isnan(x)):
        raise ValueError("fp16_ru is defined here for non-negative values only")
    with np.errstate(over="ignore"):   # above the largest binary16 the least one >= x is +inf
        h = x.astype(np.float16)
    below = h.astype(np.float64) < x
    bits = h.view(np.uint16).copy()
    bits[below] += 1            # next binary16 above a non-negative value
    return bits.view(np.float16)


def e4m3_encode(x):
    """Encode float64 values as fp8 e4m3fn bytes (RN-even, saturating)."""
    x = np.asarray(x, dtype=np.float64)
    if np.any(np.isnan(x)):
        raise ValueError("NaN input")
    sign = np.signbit(x).astype(np.uint8) << 7
    a = np.minimum(np.abs(x), E4M3_MAX)           # finite overflow saturates
    code = np.zeros(a.shape, dtype=np.uint8)

    sub = a < 2.0 ** -6                           # subnormal range: m * 2^-9
    m_sub = np.rint(a[sub] * 2.0 ** 9)            # 0..8; 8 is the least normal
    code[sub] = m_sub.astype(np.uint8)

    nor = ~sub
    _, E = np.frexp(a[nor])                       # a = f * 2^E, f in [0.5, 1)
    e = E - 1                                     # a in [2^e, 2^(e+1))
    m = np.rint(a[nor] * np.ldexp(8.0, -e)) - 8   # exact scaling, RN-even
    carry = m >= 8
    e = np.where(carry, e + 1, e)
    m = np.where(carry, 0, m)
    code[nor] = (((e + 7) << 3) | m.astype(np.int64)).astype(np.uint8)
    return code | sign


def e4m3_decode(code):
    """Exact float64 value of fp8 e4m3fn bytes (NaN for the NaN pattern)."""
    code = np.asarray(code, dtype=np.uint8)
    s = np.where(code & 0x80, -1.0, 1.0)
    E = ((code >> 3) & 0xF).astype(np.int64)
    m = (code & 0x7).astype(np.float64)
    val = np.where(E == 0, m * 2.0 ** -9, (1.0 + m / 8.0) * np.ldexp(1.0, E - 7))
    val = np.where((E == 15) & (m == 7), np.nan, val)
    return s * val
