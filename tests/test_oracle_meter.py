"""Pins for oracle.meter: paper-printed values, closed forms, brute force,
high-precision re-evaluation and invariants (no GPU)."""

import itertools
import math
import os

import mpmath
import numpy as np
import pytest

from oracle import meter as M
from oracle import quantizer as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    vals = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            k, *v = line.split()
            vals[k] = np.array([float(x) for x in v])
    return vals


def test_counterexample_matches_paper():
    g = _golden("counterexample.txt")
    p = M.perturbed(g["p_tilde"], g["eps"])
    assert np.all(np.abs(g["eps"]) <= g["c"])
    assert M.total_variation(p, g["p_tilde"]) == pytest.approx(g["true_tv"][0], abs=5e-7)
    assert M.flawed_bound(g["p_tilde"], g["c"]) == pytest.approx(g["flawed_bound"][0], abs=5e-7)
    meter, raw, A = M.eform_meter(g["p_tilde"], g["c"])
    assert raw == pytest.approx(0.5 * (math.exp(0.2) - 1.0), rel=1e-14)
    assert raw >= g["true_tv"][0] and meter == raw


def test_eform_closed_forms():
    # all c equal: A = e^c exactly, so 1/2 (A^2 - 1) = 1/2 (e^{2c} - 1)
    rng = np.random.default_rng(1)
    for c0 in [1e-9, 1e-4, 0.05, 0.7, 3.0]:
        pt = rng.dirichlet(np.ones(7))
        meter, raw, A = M.eform_meter(pt, np.full(7, c0))
        assert raw == pytest.approx(0.5 * math.expm1(2 * c0), rel=1e-12)
        assert A == pytest.approx(math.exp(c0), rel=1e-14)
        assert meter == min(1.0, raw)
    m, raw, _ = M.eform_meter(np.array([0.5, 0.5]), np.zeros(2))
    assert raw == 0.0 and m == 0.0
    m, raw, _ = M.eform_meter(np.array([1e-300, 1 - 1e-300]), np.array([800.0, 0.0]))
    assert raw == np.inf and m == 1.0
    # zero mass on a token makes its bound irrelevant, even an infinite one
    m, raw, _ = M.eform_meter(np.array([0.0, 1.0]), np.array([np.inf, 0.25]))
    assert raw == pytest.approx(0.5 * math.expm1(0.5))


def test_eform_terms_equal_the_product_on_ordinary_inputs():
    """From logits, the terms and the meter are bit for bit the product form's
    wherever float64 holds p~ and expm1(c)."""
    rng = np.random.default_rng(21)
    for S in (1, 2, 17, 300):
        z = rng.normal(0, 4, S)
        c = np.abs(rng.normal(0, 0.5, S))
        p, terms = M.eform_terms(z, c)
        assert np.array_equal(p, M.softmax(z))
        assert np.array_equal(terms, M.softmax(z) * np.expm1(c))
        for a, b in zip(M.eform_meter_logits(z, c), M.eform_meter(M.softmax(z), c)):
            assert np.array_equal(a, b)


def test_eform_terms_where_float64_underflows_or_overflows():
    """Closed forms where the product cannot be formed in float64 (§3 e-form,
    evaluated in the log domain): a weight of e^-800 / (1 + e^-800) with
    c = 801 contributes e (1 - e^-801) / (1 + e^-800) = e to D, where the
    product gives 0; a weight e^-705 / (1 + e^-705) with c = 710 contributes
    e^5, where expm1(710) overflows."""
    _, terms = M.eform_terms(np.array([0.0, -800.0]), np.array([0.0, 801.0]))
    assert terms[0] == 0.0 and terms[1] == pytest.approx(math.e, rel=1e-13)
    m, raw, A = M.eform_meter_logits(np.array([0.0, -800.0]), np.array([0.0, 801.0]))
    assert raw == pytest.approx(0.5 * math.e * (math.e + 2.0), rel=1e-13) and m == 1.0
    assert M.eform_meter(M.softmax(np.array([0.0, -800.0])), np.array([0.0, 801.0]))[1] == 0.0
    m, raw, A = M.eform_meter_logits(np.array([0.0, -705.0]), np.array([0.0, 710.0]))
    assert A - 1.0 == pytest.approx(math.exp(5.0), rel=1e-12)
    assert M.eform_meter(M.softmax(np.array([0.0, -705.0])), np.array([0.0, 710.0]))[1] == np.inf
    # beyond float64 the meter is +inf, and a zero bound adds nothing at any weight
    m, raw, _ = M.eform_meter_logits(np.array([0.0, -10.0]), np.array([0.0, 2000.0]))
    assert raw == np.inf and m == 1.0
    _, terms = M.eform_terms(np.array([0.0, -900.0]), np.array([0.25, 0.0]))
    assert terms[1] == 0.0 and terms[0] == pytest.approx(math.expm1(0.25), rel=1e-15)
    # the page contributions from these terms sum to D
    z, c = np.array([0.0, -800.0, -3.0, -790.0]), np.array([0.1, 801.0, 0.0, 792.0])
    p, terms = M.eform_terms(z, c)
    C = M.page_contributions(p, c, np.array([0, 0, 1, 1]), 2, terms=terms)
    assert C.sum() == pytest.approx(M.eform_meter_logits(z, c)[2] - 1.0, rel=1e-14)
    assert C[1] == pytest.approx(math.exp(2.0) / (1 + math.exp(-3.0)), rel=1e-12)


def test_eform_sound_against_sign_vertices_and_interior():
    """TV(p, p~) <= 1/2 (A^2 - 1) for every admissible eps (brute force)."""
    rng = np.random.default_rng(2)
    worst = 0.0
    flawed_violated = 0
    for trial in range(3000):
        S = int(rng.integers(2, 8))
        alpha = [0.05, 1.0, 20.0][trial % 3]                # peaked .. flat
        pt = rng.dirichlet(np.full(S, alpha))
        scale = [0.01, 0.3, 2.0][(trial // 3) % 3]
        c = rng.exponential(scale, S)
        eps = np.array(list(itertools.product(*[(-ci, ci) for ci in c])))
        eps = np.concatenate([eps, rng.uniform(-1, 1, (64, S)) * c])
        tv = M.total_variation(M.perturbed(pt[None, :], eps), pt[None, :])
        _, raw, _ = M.eform_meter(pt, c)
        assert np.all(tv <= raw * (1 + 1e-12) + 1e-15)
        worst = max(worst, float(np.max(tv / max(raw, 1e-300))))
        flawed_violated += int(np.any(tv > M.flawed_bound(pt, c) * (1 + 1e-9)))
    assert worst <= 1.0
    assert flawed_violated > 0        # the unsound certificate is caught


def test_tv_and_meter_at_most_one():
    rng = np.random.default_rng(3)
    for _ in range(200):
        S = 50
        pt = rng.dirichlet(np.full(S, 0.3))
        c = rng.exponential(5.0, S)
        eps = rng.choice([-1.0, 1.0], S) * c
        assert M.total_variation(M.perturbed(pt, eps), pt) <= 1.0
        meter, raw, _ = M.eform_meter(pt, c)
        assert meter <= 1.0 and meter == min(1.0, raw)


def test_softmax_tv_attention_against_mpmath():
    mpmath.mp.dps = 50
    rng = np.random.default_rng(4)
    for _ in range(5):
        S, d = 6, 4
        q = rng.normal(size=d)
        k = rng.normal(size=(S, d))
        kh = k + rng.normal(scale=0.05, size=(S, d))
        v = rng.normal(size=(S, d))

        def mp_softmax(kk):
            z = [mpmath.fsum(mpmath.mpf(q[i]) * mpmath.mpf(kk[t, i]) for i in range(d)) / mpmath.sqrt(d)
                 for t in range(S)]
            e = [mpmath.exp(x) for x in z]
            tot = mpmath.fsum(e)
            return [x / tot for x in e]

        p, pt = mp_softmax(k), mp_softmax(kh)
        tv = mpmath.fsum(abs(a - b) for a, b in zip(p, pt)) / 2
        y = [mpmath.fsum(pt[t] * mpmath.mpf(v[t, i]) for t in range(S)) for i in range(d)]
        po, pto = M.softmax(M.logits(q, k)), M.softmax(M.logits(q, kh))
        assert np.allclose(po, [float(x) for x in p], rtol=1e-13, atol=0)
        assert M.total_variation(po, pto) == pytest.approx(float(tv), rel=1e-10)
        assert np.allclose(M.attend(pto, v), [float(x) for x in y], rtol=1e-12, atol=1e-14)


def _pairs(layout, d=128):
    j = np.arange(d // 2)
    if layout == Q.ROPE_HALF:
        return np.stack([j, j + d // 2], axis=1)
    if layout == Q.ROPE_INTERLEAVED:
        return np.stack([2 * j, 2 * j + 1], axis=1)
    # a pairing that crosses bands, used as a negative control
    return np.stack([np.arange(0, d, 2), np.roll(np.arange(1, d, 2), 9)], axis=1)


def _rope_rotate(x, n, pairs, theta=1e4):
    """Rotate x [d] by position n in fp64: pair j turns by n * theta^(-2j/d)."""
    d = x.shape[-1]
    ang = n * theta ** (-2.0 * np.arange(len(pairs)) / d)
    a, b = x[pairs[:, 0]], x[pairs[:, 1]]
    y = x.copy()
    y[pairs[:, 0]] = a * np.cos(ang) - b * np.sin(ang)
    y[pairs[:, 1]] = a * np.sin(ang) + b * np.cos(ang)
    return y


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
def test_band_norms_rope_invariant(layout):
    """Lemma "RoPE band unitarity": band norms do not change under R_n."""
    rng = np.random.default_rng(5)
    moved = 0
    for _ in range(20):
        r = rng.normal(size=128) * np.exp(rng.normal(size=128))
        n = int(rng.integers(1, 131072))
        rr = _rope_rotate(r, n, _pairs(layout))
        assert np.allclose(Q.band_norms(rr, 8, layout), Q.band_norms(r, 8, layout), rtol=1e-12)
        wrong = _rope_rotate(r, n, _pairs(-1))
        moved += int(not np.allclose(Q.band_norms(wrong, 8, layout),
                                     Q.band_norms(r, 8, layout), rtol=1e-6))
    assert moved > 0      # a pairing that crosses bands is detected
    # every dim belongs to exactly one band, and every pair lies in one band
    dims = Q.band_dims(128, 8, layout)
    assert sorted(dims.reshape(-1).tolist()) == list(range(128))
    band_of = np.empty(128, int)
    for b in range(8):
        band_of[dims[b]] = b
    P = _pairs(layout)
    assert np.all(band_of[P[:, 0]] == band_of[P[:, 1]])


def test_tier_a_bound_cauchy_schwarz():
    rng = np.random.default_rng(6)
    for layout in (Q.ROPE_HALF, Q.ROPE_INTERLEAVED):
        dims = Q.band_dims(128, 8, layout)
        for _ in range(50):
            r = rng.normal(size=(5, 128)) * 0.01
            w = Q.band_norms(r, 8, layout)
            q = rng.normal(size=128) * 3
            c = M.tier_a_bound(q, w, 8, layout)
            assert np.all(np.abs(r @ q) / math.sqrt(128) <= c * (1 + 1e-12))
            # adversarial query: q_b parallel to r_b for token 0 -> equality
            lam = rng.uniform(0.5, 2.0, 8)
            qa = np.zeros(128)
            for b in range(8):
                qa[dims[b]] = lam[b] * r[0, dims[b]]
            ca = M.tier_a_bound(qa, w, 8, layout)
            assert ca[0] == pytest.approx(abs(r[0] @ qa) / math.sqrt(128), rel=1e-12)


def test_gate_definition():
    mr = np.array([0.0, 0.1, np.float32(0.1) + 1e-7, np.inf, np.nan, 0.05, 0.2, 0.3], np.float32)
    keep_q, keep_kv, nq, nkv = M.gate(mr, 0.1, 2)
    assert keep_q.tolist() == [True, True, False, False, False, True, False, False]
    assert keep_kv.tolist() == [True, False, False, False]
    assert (nq, nkv) == (3, 1)
