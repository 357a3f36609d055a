"""Pins for the oracle's block-level repair selection (§6.3.5 "Block-level
paging"): the certificate is block decomposable, so paging in page j (its
exact keys carry a zero witness) lowers A by exactly that page's contribution
C_j with p~ held fixed; the plan is the fewest pages that bring the meter to
tau, checked by brute force over all page subsets; and the edge cases
(nothing to repair, tau < 0, non-finite contributions, ties, GQA groups)."""

import itertools

import numpy as np
import pytest

import workloads as W
from oracle import meter as M
from oracle import pipeline as OP


def _setup(ctx_lens, seed=3, scheme=OP.SCHEME_DITHER_INT8):
    wl = W.Workload("r", 1, 8, 2, ctx_lens, shuffle_pages=True, seed=seed)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, 0)
    q = W.layer_queries(wl, 0).numpy()
    od = OP.Desc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=scheme, seed=9)
    cache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k.numpy(), v.numpy(), sm, cache)
    return od, cache, bt, q


def _with_exact_pages(od, cache, bt_row, kv_head, pages):
    """A copy of the cache in which the given logical pages of one KV head hold
    exact keys as far as the meter is concerned: their witness is zero."""
    c2 = {k: np.array(v, copy=True) for k, v in cache.items()}
    for j in pages:
        c2["k_witness"][bt_row[j], kv_head] = 0
    return c2


@pytest.mark.parametrize("scheme", [OP.SCHEME_DITHER_INT8, OP.SCHEME_FP8_E4M3])
def test_paging_in_a_page_lowers_A_by_its_contribution(scheme):
    od, cache, bt, q = _setup([203], scheme=scheme)
    S = 203
    r = OP.decode_sequence(od, 0, q[0] * 3.0, bt[0], S, cache, repair_tau=0.0)
    n_pages = (S + 15) // 16
    assert r["contrib"].shape == (8, n_pages)
    for hq in (0, 5):
        h = hq // 4
        for j in (0, 6, n_pages - 1):                  # first, middle, ragged last page
            r2 = OP.decode_sequence(od, 0, q[0] * 3.0, bt[0], S, _with_exact_pages(od, cache, bt[0], h, [j]))
            assert r["A"][hq] - r2["A"][hq] == pytest.approx(r["contrib"][hq, j], rel=1e-9, abs=1e-15)
            # the other KV head's query heads are untouched
            other = 4 * (1 - h)
            assert r2["A"][other] == r["A"][other]


def test_shared_radius_gives_mass_times_expm1():
    # a block whose tokens share one radius u_j contributes mass_j (e^{u_j} - 1)
    rng = np.random.default_rng(4)
    S, P = 100, 16
    p_t = M.softmax(rng.standard_normal(S) * 2)
    page = np.arange(S) // P
    u = rng.uniform(0.0, 0.3, page.max() + 1)
    C = M.page_contributions(p_t, u[page], page, page.max() + 1)
    mass = np.array([p_t[page == j].sum() for j in range(page.max() + 1)])
    np.testing.assert_allclose(C, mass * np.expm1(u), rtol=1e-12)


def _meter_after(C, taken):
    R = sum(C[j] for j in range(len(C)) if j not in set(taken))
    return 0.5 * R * (R + 2.0)


def test_plan_is_the_fewest_pages_bruteforce():
    rng = np.random.default_rng(5)
    for trial in range(300):
        n = int(rng.integers(1, 9))
        C = rng.exponential(0.05, n) * (rng.random(n) < 0.8)
        D = C.sum()
        tau = float(rng.uniform(0, 0.5 * D * (D + 2.0) * 1.2)) if D > 0 else 0.0
        plan, R = M.repair_plan(C, tau)
        assert _meter_after(C, plan) <= tau * (1 + 1e-12) + 1e-300
        assert R == pytest.approx(sum(C[j] for j in range(n) if j not in plan), abs=1e-15)
        need = min(len(s) for k in range(n + 1) for s in itertools.combinations(range(n), k)
                   if _meter_after(C, s) <= tau)
        assert len(plan) == need, (C, tau, plan)
        assert all(C[a] >= C[b] for a, b in zip(plan, plan[1:]))


def test_plan_edge_cases():
    assert M.repair_plan(np.zeros(0), 0.1) == ([], 0.0)
    assert M.repair_plan(np.array([0.01, 0.02]), 0.1)[0] == []         # already below tau
    assert M.repair_plan(np.array([0.01, 0.02]), -1.0)[0] == [1, 0]    # tau < 0: every page
    plan, R = M.repair_plan(np.array([0.01, np.inf, 0.02, np.inf]), 0.1)
    assert plan == [1, 3] and R == pytest.approx(0.03)
    plan, R = M.repair_plan(np.array([0.3, np.nan, 0.01]), 0.1)
    assert plan == [1, 0] and R == pytest.approx(0.01)
    assert M.repair_plan(np.array([0.2, 0.2, 0.2, 0.0]), 0.3)[0] == [0, 1]   # ties: lower page first
    # the threshold in exact binary values: 1/2 R (R + 2) = tau keeps (R = 0.25, tau = 0.28125)
    assert M.repair_plan(np.array([0.25, 0.5]), 0.28125) == ([1], 0.25)
    assert M.repair_plan(np.array([0.25, 0.5]), np.nextafter(0.28125, 0.0)) == ([1, 0], 0.0)


@pytest.mark.parametrize("scale", [2.0, 4.0])
def test_plan_repairs_through_the_pipeline_and_is_minimal(scale):
    od, cache, bt, q = _setup([300, 91], seed=6)
    for b, S in enumerate([300, 91]):
        base = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S, cache)
        for hq in (1, 6):
            tau = base["meter_raw"][hq] / 4.0
            r = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S, cache, repair_tau=tau)
            plan = r["repair"][hq]
            assert len(plan) >= 1
            h = hq // 4
            fixed = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S, _with_exact_pages(od, cache, bt[b], h, plan))
            assert fixed["meter_raw"][hq] <= tau * (1 + 1e-9)
            short = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S,
                                       _with_exact_pages(od, cache, bt[b], h, plan[:-1]))
            assert short["meter_raw"][hq] > tau


def test_union_of_a_group_repairs_every_head():
    od, cache, bt, q = _setup([250], seed=8)
    base = OP.decode_sequence(od, 0, q[0] * 3.0, bt[0], 250, cache)
    tau = float(np.median(base["meter_raw"])) / 3.0
    r = OP.decode_sequence(od, 0, q[0] * 3.0, bt[0], 250, cache, repair_tau=tau)
    for h in range(2):
        union = sorted(set().union(*[r["repair"][hq] for hq in range(4 * h, 4 * h + 4)]))
        fixed = OP.decode_sequence(od, 0, q[0] * 3.0, bt[0], 250, _with_exact_pages(od, cache, bt[0], h, union))
        assert np.all(fixed["meter_raw"][4 * h:4 * h + 4] <= tau * (1 + 1e-9))
