"""Pins for oracle.fp and oracle.quantizer: exact rational arithmetic,
torch's own casts (a library), and the quantizer's stated guarantees."""

import math
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import fp, quantizer as Q
from oracle import philox

ALL_FP16 = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16).view(np.float16)
FINITE = ALL_FP16[np.isfinite(ALL_FP16)]


def _fp16_grid_neighbours(x):
    """Exact fp16 values just below/above x (as Fractions) by bisection."""
    pos = np.sort(np.unique(FINITE[FINITE >= 0].astype(np.float64)))
    i = np.searchsorted(pos, x)
    return pos[max(i - 1, 0)], pos[min(i, len(pos) - 1)]


def test_fp16_rn_matches_exact_nearest_even():
    rng = np.random.default_rng(10)
    xs = np.concatenate([rng.uniform(0, 70000, 2000), np.exp(rng.uniform(-20, 11, 2000))])
    pos = np.sort(np.unique(FINITE[FINITE >= 0].astype(np.float64)))
    # plus exact midpoints between neighbours (ties)
    mids = (pos[:-1][::97] + pos[1:][::97]) / 2
    for x in np.concatenate([xs[xs < 65504], mids]):
        i = np.searchsorted(pos, x)
        lo, hi = pos[i - 1] if pos[i] != x else pos[i], pos[i]
        dl, dh = Fraction(x) - Fraction(lo), Fraction(hi) - Fraction(x)
        if dl < dh:
            want = lo
        elif dh < dl:
            want = hi
        else:
            want = lo if (np.float16(lo).view(np.uint16) % 2 == 0) else hi
        assert float(fp.fp16_rn(x)) == want


def test_fp16_ru_is_least_upper_fp16():
    rng = np.random.default_rng(11)
    xs = np.exp(rng.uniform(-25, 11, 5000))
    xs = xs[xs < 65504]
    up = fp.fp16_ru(xs).astype(np.float64)
    assert np.all(up >= xs)
    below = (fp.fp16_ru(xs).view(np.uint16) - 1).view(np.float16).astype(np.float64)
    assert np.all((below < xs) | (up == xs))
    assert float(fp.fp16_ru(0.0)) == 0.0
    assert float(fp.fp16_ru(1e-12)) == 2.0 ** -24


def test_e4m3_exhaustive_against_torch():
    x = FINITE[np.abs(FINITE.astype(np.float64)) < 464]
    mine = fp.e4m3_encode(x.astype(np.float64))
    ref = torch.from_numpy(x.copy()).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(mine, ref)
    codes = np.arange(256, dtype=np.uint8)
    dec = fp.e4m3_decode(codes)
    tdec = torch.from_numpy(codes).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    both_nan = np.isnan(dec) & np.isnan(tdec)
    assert np.array_equal(dec[~both_nan], tdec[~both_nan]) and np.array_equal(np.isnan(dec), np.isnan(tdec))


def test_e4m3_saturates():
    big = np.array([448.0, 463.9, 464.0, 465.0, 1e4, 65504.0])
    assert np.all(fp.e4m3_decode(fp.e4m3_encode(big)) == 448.0)
    assert np.all(fp.e4m3_decode(fp.e4m3_encode(-big)) == -448.0)


def test_scale_matches_torch_fp32_division_then_fp16():
    amax = FINITE[FINITE > 0]
    rows = np.zeros((amax.size, 4), np.float16)
    rows[:, 1] = -amax
    s = Q.int8_scale(rows)
    ref = (torch.from_numpy(amax.copy()).float() / 126.5).half().numpy()
    ref = np.where(ref == 0, np.float16(2.0 ** -24), ref)
    assert np.array_equal(s.view(np.uint16), ref.view(np.uint16))
    assert Q.int8_scale(np.zeros((1, 8), np.float16))[0] == 0


def _xi_grid(bits, n, rng):
    return philox.dither_values(rng.integers(0, 1 << bits, n), bits)


@pytest.mark.parametrize("bits", [8, 10])
def test_dither_code_matches_fraction_rounding(bits):
    rng = np.random.default_rng(12)
    n = 4000
    x = rng.normal(size=n).astype(np.float16) * np.float16(3)
    s = Q.int8_scale(x.reshape(-1, 40)).repeat(40)
    xi = _xi_grid(bits, n, rng)
    got = Q.dither_code(x.reshape(-1, 40), s.reshape(-1, 40)[:, 0], xi.reshape(-1, 40)).reshape(-1)
    for i in range(n):
        assert got[i] == Q.dither_code_fraction(x[i], s[i], xi[i])
    # random (x, s) pairs including clipping scales and subnormals
    x2 = rng.choice(FINITE, 3000)
    s2 = np.abs(rng.choice(FINITE, 3000))
    xi2 = _xi_grid(bits, 3000, rng)
    got2 = Q.dither_code(x2[:, None], s2, xi2[:, None])[:, 0]
    for i in range(3000):
        assert got2[i] == Q.dither_code_fraction(x2[i], s2[i], xi2[i])


@pytest.mark.parametrize("bits", [8, 10])
def test_dither_code_ties_go_to_even(bits):
    # x = s (k + 1/2 - xi) exactly: choose s = 2^-e and small k so x is fp16
    rng = np.random.default_rng(13)
    count = 0
    for _ in range(4000):
        j = int(rng.integers(0, 1 << bits))
        xi = (j + 0.5) / (1 << bits) - 0.5
        k = int(rng.integers(-3, 3))
        e = int(rng.integers(0, 4))
        s = 2.0 ** -e
        x = s * (k + 0.5 - xi)
        if float(np.float16(x)) != x:
            continue
        code = Q.dither_code(np.array([[x]], np.float16), np.array([s], np.float16), np.array([[xi]]))[0, 0]
        assert code == (k if k % 2 == 0 else k + 1)
        count += 1
    assert count > 500


@pytest.mark.parametrize("bits", [8, 10])
def test_no_clipping_and_half_step_error(bits):
    """s = amax / 126.5 leaves no clipping and |x^ - x| <= s / 2 exactly."""
    rng = np.random.default_rng(14)
    rows = (rng.normal(size=(3000, 128)) * np.exp(rng.normal(size=(1, 128)))).astype(np.float16)
    rows[::7] *= np.float16(100)
    s = Q.int8_scale(rows)
    xi = _xi_grid(bits, rows.size, rng).reshape(rows.shape)
    code = Q.dither_code(rows, s, xi)
    y_exact_max = np.max(np.abs(rows.astype(np.float64) / s.astype(np.float64)[:, None] + xi), axis=1)
    assert np.all(y_exact_max < 127.5)                     # never clipped
    err = Q.dither_reconstruct(code, s, xi) - rows.astype(np.float64)
    assert np.all(np.abs(err) <= s.astype(np.float64)[:, None] / 2)
    assert np.max(np.abs(err) / (s.astype(np.float64)[:, None] / 2)) > 0.99


def _ru16_of_sqrt_exact(sumsq):
    """Least fp16 h >= sqrt(sumsq) for an exact Fraction sumsq."""
    approx = math.sqrt(float(sumsq))
    cand = float(fp.fp16_ru(approx))
    h = np.float16(cand)
    while Fraction(float(h)) ** 2 < sumsq:
        h = (np.array([h]).view(np.uint16) + 1).view(np.float16)[0]
    while True:
        prev = (np.array([h]).view(np.uint16) - 1).view(np.float16)[0]
        if float(h) > 0 and Fraction(float(prev)) ** 2 >= sumsq:
            h = prev
        else:
            return float(h)


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
def test_witness_is_rounded_up_exact_band_norm(layout):
    rng = np.random.default_rng(15)
    rows = (rng.normal(size=(40, 128)) * 2).astype(np.float16)
    s = Q.int8_scale(rows)
    xi = _xi_grid(8, rows.size, rng).reshape(rows.shape)
    code = Q.dither_code(rows, s, xi)
    resid = Q.dither_reconstruct(code, s, xi) - rows.astype(np.float64)
    w = Q.witness(resid, 8, layout)
    dims = Q.band_dims(128, 8, layout)
    for t in range(rows.shape[0]):
        for b in range(8):
            exact = sum(Fraction(float(s[t])) ** 2 * (Fraction(int(code[t, d])) - Fraction(float(xi[t, d]))) ** 2
                        - 2 * Fraction(float(s[t])) * (Fraction(int(code[t, d])) - Fraction(float(xi[t, d])))
                        * Fraction(float(rows[t, d])) + Fraction(float(rows[t, d])) ** 2
                        for d in dims[b])
            assert float(w[t, b]) == _ru16_of_sqrt_exact(exact)


def test_fp8_zero_residual_gives_zero_witness():
    codes = np.arange(0, 0x7F, dtype=np.uint8)
    vals = fp.e4m3_decode(codes)
    row = np.resize(vals, 128).astype(np.float16)          # e4m3 values are fp16-exact
    code, rec = Q.fp8_quantize(row[None, :])
    assert np.array_equal(rec[0], row.astype(np.float64))
    assert np.all(Q.witness(rec - row.astype(np.float64), 8, Q.ROPE_HALF) == 0)
