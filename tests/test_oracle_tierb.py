"""Pins for the oracle's Tier-B certificate (§4.2): the Lemma's inequality,
the sub-Gaussian proxy against the quantizer's measured logit-error variance
over dither seeds, zero-violation counting for fixed (non-adaptive) queries,
and the degenerate cases.  None of these re-derives the oracle's formula."""

import numpy as np
import pytest

from oracle import meter as M
from oracle import pipeline as OP


def test_lemma_uniform_mgf_bounded_by_gaussian():
    """E[e^{lX}] = sinh(la)/(la) <= e^{l^2 a^2/6} for X ~ U[-a, a] (Lemma)."""
    x = np.concatenate([np.logspace(-4, 1.6, 400), [1.0, 2.0, 5.0]])
    assert np.all(np.sinh(x) / x <= np.exp(x * x / 6) * (1 + 1e-15))
    # the closed-form MGF itself, against a Monte-Carlo estimate
    rng = np.random.default_rng(0)
    a, lam = 0.7, 1.9
    X = rng.uniform(-a, a, size=2_000_000)
    assert abs(np.mean(np.exp(lam * X)) - np.sinh(lam * a) / (lam * a)) < 2e-3


def _rows(rng, n, d=128):
    return (rng.standard_normal((n, d)) * rng.lognormal(0, 0.5, size=d)).astype(np.float16)


def test_proxy_equals_measured_logit_error_variance():
    """Over dither seeds the logit error q . r_t / sqrt(d) has variance
    ||q||^2 s_t^2 / (12 d); the oracle's u_t encodes exactly that proxy."""
    rng = np.random.default_rng(1)
    k = _rows(rng, 8)
    q = rng.standard_normal(128)
    slots = np.arange(8)
    errs = []
    for seed in range(1500):
        desc = OP.Desc(num_kv_heads=1, num_q_heads=1, seed=seed)
        _, s, khat = OP.quantize_rows(desc, 3, 0, k, slots, 0)
        errs.append((khat - k.astype(np.float64)) @ q / np.sqrt(128))
    errs = np.array(errs)                                    # [seeds, tokens]
    u = M.tier_b_bound(q, s.astype(np.float64), ctx_len=8, delta_loc=0.05)
    proxy = u * u / (2 * np.log(2 * 8 / 0.05))              # varsigma_t^2
    measured = errs.var(axis=0)
    # sample variance of 1500 draws: relative standard error ~ sqrt(2/1500) = 3.7%
    assert np.all(np.abs(measured / proxy - 1) < 0.15), measured / proxy
    assert np.all(np.abs(errs.mean(axis=0)) < 4 * np.sqrt(proxy / 1500))   # subtractive dither: unbiased


def test_zero_violations_for_fixed_queries():
    """Non-adaptive queries: over dither seeds, |eps_t| <= u_t for all tokens
    fails with probability <= delta_loc; whenever it holds, TV <= meter_b."""
    rng = np.random.default_rng(2)
    S, delta = 48, 0.05
    k = _rows(rng, S)
    k[0] *= 8                                                  # sink token
    qs = rng.standard_normal((4, 128)) * np.array([[1.0], [2.0], [4.0], [8.0]])
    slots = np.arange(S)
    seeds_with_violation = 0
    for seed in range(120):
        desc = OP.Desc(num_kv_heads=1, num_q_heads=4, seed=1000 + seed)
        _, s, khat = OP.quantize_rows(desc, 0, 0, k, slots, 0)
        viol = False
        for q in qs:
            eps = (khat - k.astype(np.float64)) @ q / np.sqrt(128)
            u = M.tier_b_bound(q, s.astype(np.float64), S, delta)
            p_t = M.softmax(M.logits(q, khat))
            p = M.softmax(M.logits(q, k.astype(np.float64)))
            if np.all(np.abs(eps) <= u):
                assert M.total_variation(p, p_t) <= M.eform_meter(p_t, u)[1] * (1 + 1e-12)
            else:
                viol = True
        seeds_with_violation += viol
    # 4 queries per seed: at most 4 * delta of the seeds may fail (union bound)
    assert seeds_with_violation <= 4 * delta * 120


def test_degenerate_cases():
    q = np.linspace(-1, 1, 128)
    s = np.array([0.0, 0.01, 0.02])
    u = M.tier_b_bound(q, s, 3, 0.01)
    assert u[0] == 0.0
    assert u[2] == pytest.approx(2 * u[1], rel=1e-12)                        # linear in s
    assert M.tier_b_bound(3 * q, s, 3, 0.01)[1] == pytest.approx(3 * u[1])   # linear in ||q||
    assert M.tier_b_bound(q, s, 3, 0.001)[1] > u[1]                          # tighter delta, larger u
    # an all-zero cache row (s = 0) contributes nothing to the meter
    _, raw, _ = M.eform_meter(np.array([0.5, 0.5]), np.array([0.0, 0.0]))
    assert raw == 0.0


def test_decode_sequence_tier_b_only_for_the_dithered_cache():
    desc = OP.Desc(num_kv_heads=1, num_q_heads=2, num_pages=2, scheme=OP.SCHEME_FP8_E4M3)
    cache = OP.empty_cache(desc)
    with pytest.raises(ValueError):
        OP.decode_sequence(desc, 0, np.zeros((2, 128), np.float16), np.array([0, 1]), 20, cache, delta_loc=0.01)
