"""The exponent the decode kernels use for a meter term with a huge bound,
checked on the CPU in the kernels' fp32 evaluation order.

For a token with weight 2^t in the log2 frame of the running maximum and a
bound cl = c log2(e) of 2^64 or more, the term p~ (e^c - 1) = 2^t (2^cl - 1) is
taken as 2^e with e = fp32(fp32(t + cl) + fp32(fp32(|t| + cl) * 2^-22)).  That
e must never be below the exact t + cl (the term is then never under-counted),
and its excess must stay small enough that 2^e is within the parity tolerance
of the term: at most (|t| + cl) 2^-21, i.e. a relative excess of at most
(|t| + cl) 2^-21 ln 2: below 2^-12 while |t| + cl < 512 and below the 1e-3
parity tolerance while |t| + cl < 3000."""

from fractions import Fraction

import numpy as np

F = np.float32


def exponent(t, cl):
    t, cl = F(t), F(cl)
    s = F(t + cl)
    m = F(F(abs(t) + cl) * F(2.0 ** -22))
    return F(s + m)


def _cases():
    r = np.random.default_rng(11)
    ts = np.concatenate([-r.uniform(0, 2000, 4000), -r.uniform(0, 300, 4000), r.uniform(-130, 0, 2000),
                         -np.exp(r.uniform(0, 14, 2000))]).astype(np.float32)
    cls = np.concatenate([r.uniform(64, 2000, 4000), r.uniform(64, 300, 4000), r.uniform(64, 140, 2000),
                          np.exp(r.uniform(np.log(64), 14, 2000))]).astype(np.float32)
    # near-cancellation: cl just above -t, and the smallest bound the path takes
    near = -ts[:3000] + r.uniform(-3, 3, 3000).astype(np.float32)
    ts = np.concatenate([ts, ts[:3000], -r.uniform(0, 200, 500).astype(np.float32)])
    cls = np.concatenate([cls, np.maximum(near, 64).astype(np.float32), np.full(500, 64, np.float32)])
    return ts, cls


def test_raised_exponent_is_never_below_the_exact_sum():
    ts, cls = _cases()
    for t, cl in zip(ts, cls):
        e = exponent(t, cl)
        exact = Fraction(float(t)) + Fraction(float(cl))
        assert Fraction(float(e)) >= exact, (float(t), float(cl))


def test_raised_exponent_excess_is_small():
    ts, cls = _cases()
    for t, cl in zip(ts, cls):
        e = exponent(t, cl)
        exact = Fraction(float(t)) + Fraction(float(cl))
        excess = Fraction(float(e)) - exact
        assert excess <= (abs(Fraction(float(t))) + Fraction(float(cl))) * Fraction(1, 2 ** 21), \
            (float(t), float(cl), float(excess))


def test_relative_excess_of_the_term():
    ts, cls = _cases()
    size = np.abs(ts.astype(np.float64)) + cls
    for t, cl, n in zip(ts, cls, size):
        excess = float(Fraction(float(exponent(t, cl))) - Fraction(float(t)) - Fraction(float(cl)))
        rel = 2.0 ** excess - 1.0
        if n < 512:
            assert rel < 2.0 ** -12, (float(t), float(cl))
        if n < 3000:
            assert rel < 1e-3, (float(t), float(cl))
