"""GPU parity of block-level repair selection (§6.3.5 "Block-level paging"):
the decode with per-page terms leaves the plain outputs bit for bit, the page
contributions C_j match the oracle's, the list is consistent with the
kernel's own contributions (ordering; the count may differ only where the
meter sits within rounding of tau), the chosen pages are a top set of the oracle's fp64
contributions that brings the meter to tau, and the edge cases (kept cells,
NaN / inf / tied / zero contributions, ragged and one-token contexts, the
largest block table) select what the oracle selects."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from tests._parity import assert_close, descs, make_inputs, numpy_cache_to_gpu

pytestmark = pytest.mark.gpu


def _remaining_meter(C, taken):
    mask = np.ones(len(C), bool)
    mask[list(taken)] = False
    R = float(np.sum(C[mask]))
    return R, 0.5 * R * (R + 2.0)


def _self_order(c64):
    """The ranking rule applied to the kernel's own contributions (a check of
    the selection kernel's consistency, not an oracle result): NaN first, then
    by decreasing contribution, ties to the lower page."""
    key = np.where(np.isnan(c64), np.inf, c64)
    nan_first = np.isnan(c64)
    return sorted(range(len(c64)), key=lambda j: (not nan_first[j], -key[j], j))


def _check_selection(gc, pages, n, d_after, tau, ref_c=None):
    """One flagged cell: gc the kernel's contributions (fp32) of its n pages.
    The list is checked for consistency with the kernel's own contributions
    (ordering and the least count whose remaining meter is at most tau), and
    against the oracle's fp64 contributions ref_c (a top set that repairs)."""
    c64 = gc.astype(np.float64)
    k = len(pages)
    order = _self_order(c64)
    assert list(pages) == order[:k]                             # ranked by the kernel's own values
    rest = float(np.sum(c64)) - np.concatenate([[0.0], np.cumsum(c64[order])])   # R after i pages
    ok = np.nonzero(0.5 * rest * (rest + 2.0) <= tau)[0]
    need = int(ok[0]) if ok.size else n
    if k != need:                                               # only at the decision boundary
        _, raw = _remaining_meter(c64, order[:min(k, need)])
        assert abs(k - need) == 1 and abs(raw - tau) <= 1e-5 * max(tau, 1e-3), (k, need, raw, tau)
    R, _ = _remaining_meter(c64, pages)
    assert abs(d_after - R) <= 1e-5 * max(R, 1e-6) + 1e-7
    if ref_c is not None and 0 < k < n:                         # against the oracle's own contributions
        tol = 1e-3 * float(np.max(ref_c)) + 1e-7
        chosen = ref_c[list(pages)]
        rest = np.delete(ref_c, list(pages))
        assert chosen.min() >= rest.max() - tol                 # a top-k set
        _, raw = _remaining_meter(ref_c, pages)
        assert raw <= tau * (1 + 2e-3) + 1e-6                   # and it repairs


@pytest.mark.parametrize("scheme,bits", [(0, 8), (0, 10), (1, 8)])
def test_repair_terms_and_selection_against_oracle(scheme, bits):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("r", 1, 28, 4, [4100, 77, 1, 2500, 16, 999], shuffle_pages=True, seed=11)
    layer = 2
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, scheme, bits, 0, 5)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    res = wc.metered_decode_attention_repair(gd, layer, qd, btd, ctx, gcache, ws)
    plain = wc.metered_decode_attention(gd, layer, qd, btd, ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    for x, y in zip(plain, res[:3]):
        assert torch.equal(x, y)                                # the plain outputs are untouched
    meter_raw = res[2].cpu().numpy()
    tau = float(np.median(meter_raw)) * 0.6
    keep_q, _, _ = wc.gate(res[2].reshape(-1), gd.group, tau)
    contrib, pages, n_rep, d_after = wc.repair_select(res[3], res[4], ctx, tau, keep_q=keep_q)
    # every cell selected, contributions not stored
    _, pages_all, n_all, _ = wc.repair_select(res[3], res[4], ctx, tau, contrib=False)
    torch.cuda.synchronize()
    contrib, pages, n_rep, d_after = (t.cpu().numpy() for t in (contrib, pages, n_rep, d_after))
    keep = keep_q.cpu().numpy().reshape(wl.batch, -1).astype(bool)
    n_all, pages_all = n_all.cpu().numpy(), pages_all.cpu().numpy()
    flagged = 0
    for b, S in enumerate(wl.ctx_lens):
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, repair_tau=tau)
        n = (S + 15) // 16
        assert_close(contrib[b, :, :n], r["contrib"], f"contrib[{b}]", atol=1e-6)
        D = np.sqrt(1.0 + 2.0 * meter_raw[b].astype(np.float64)) - 1.0
        assert_close(contrib[b, :, :n].astype(np.float64).sum(axis=1), D, f"sum contrib[{b}]", atol=1e-6)
        for hq in range(wl.n_q_heads):
            if keep[b, hq]:
                assert n_rep[b, hq] == 0
                assert abs(d_after[b, hq] - contrib[b, hq, :n].astype(np.float64).sum()) <= 1e-5 * D[hq] + 1e-7
            else:
                flagged += 1
                _check_selection(contrib[b, hq, :n], pages[b, hq, :n_rep[b, hq]], n, d_after[b, hq], tau,
                                 r["contrib"][hq])
            # with keep_q absent every cell gets its list; flagged cells agree
            if not keep[b, hq]:
                assert n_all[b, hq] == n_rep[b, hq]
                assert np.array_equal(pages_all[b, hq, :n_all[b, hq]], pages[b, hq, :n_rep[b, hq]])
    assert flagged > 0


def _terms_from_contributions(C_rows, max_pages):
    """page_terms with m_j = 0 and (M, L) = (0, 1): then C_j = d_j exactly."""
    cells = len(C_rows)
    pt = np.zeros((1, cells, max_pages, 2), np.float32)
    for i, C in enumerate(C_rows):
        pt[0, i, :len(C), 1] = C
    norm = np.zeros((1, cells, 2), np.float32)
    norm[..., 1] = 1.0
    return torch.from_numpy(pt).cuda(), torch.from_numpy(norm).cuda()


@pytest.mark.parametrize("max_pages", [1, 5, 512, 513, 2048, 16384])
def test_selection_edge_cases_exact(max_pages):
    import paper_2607_28699_gb300 as wc
    rng = np.random.default_rng(max_pages)
    n = max_pages
    rows = [
        rng.exponential(1e-3, n).astype(np.float32),                                 # many small pages
        (rng.exponential(1e-3, n) * (rng.random(n) < 0.1)).astype(np.float32),        # mostly zero
        np.full(n, 2e-3, np.float32),                                                # all tied
        rng.exponential(1e-3, n).astype(np.float32),
        np.zeros(n, np.float32),
    ]
    rows[3][rng.integers(0, n)] = np.inf
    if n > 2:
        rows[3][rng.integers(0, n)] = np.nan
    rows[1][0] = -0.0
    pt, norm = _terms_from_contributions(rows, max_pages)
    ctx = torch.tensor([16 * n], dtype=torch.int32, device="cuda")
    for tau in (0.0, 0.01, 0.1, 10.0, -1.0):
        contrib, pages, n_rep, d_after = wc.repair_select(pt, norm, ctx, tau)
        torch.cuda.synchronize()
        contrib, pages, n_rep, d_after = (t.cpu().numpy() for t in (contrib, pages, n_rep, d_after))
        for i, C in enumerate(rows):
            C = C.astype(np.float32)
            C[C <= 0] = 0.0                                                          # -0 is +0
            got = contrib[0, i]
            assert np.array_equal(got.view(np.uint32)[~np.isnan(C)], C.view(np.uint32)[~np.isnan(C)])
            assert np.array_equal(np.isnan(got), np.isnan(C))
            k = n_rep[0, i]
            plan, R = OM.repair_plan(C.astype(np.float64), tau)
            order, _ = OM.repair_plan(C.astype(np.float64), -1.0)
            assert list(pages[0, i, :k]) == order[:k]
            if k != len(plan):                                                       # only at the boundary
                Rm, raw = _remaining_meter(C.astype(np.float64), order[:min(k, len(plan))])
                assert abs(k - len(plan)) == 1 and abs(raw - tau) <= 1e-5 * max(abs(tau), 1e-3)
            else:
                assert d_after[0, i] == pytest.approx(R, rel=1e-5, abs=1e-7) or (np.isnan(R) and np.isnan(d_after[0, i]))


def test_selection_short_context_and_kept_cells():
    import paper_2607_28699_gb300 as wc
    C = np.array([0.05, 0.2, 0.01, 0.3], np.float32)
    pt, norm = _terms_from_contributions([C, C], 8)
    ctx = torch.tensor([33], dtype=torch.int32, device="cuda")   # 3 pages: the 4th is past the context
    keep = torch.tensor([[0, 1]], dtype=torch.uint8, device="cuda")
    contrib, pages, n_rep, d_after = wc.repair_select(pt, norm, ctx, 0.011, keep_q=keep)   # R = 0.01 passes
    torch.cuda.synchronize()
    assert n_rep.cpu().tolist() == [[2, 0]]
    assert pages[0, 0, :2].cpu().tolist() == [1, 0]
    assert d_after.cpu().numpy()[0] == pytest.approx([0.01, 0.26], rel=1e-6)
    assert contrib[0, 0, :3].cpu().tolist() == pytest.approx([0.05, 0.2, 0.01])
    assert np.all(contrib[0, :, 3:].cpu().numpy() == 0)          # past the context: not written


def test_layers_stacked_along_batch_select_as_separate_calls():
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("s", 2, 8, 2, [700, 160, 33], shuffle_pages=True, seed=13)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, 0, 8, 0, 3)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    terms, norms, raws = [], [], []
    for layer in range(2):
        bt, sm, k, v, q = make_inputs(wl, layer)
        cache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
        res = wc.metered_decode_attention_repair(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx, cache, ws)
        terms.append(res[3]); norms.append(res[4]); raws.append(res[2])
    tau = float(torch.cat(raws).median()) * 0.5
    stacked = wc.repair_select(torch.cat(terms), torch.cat(norms), ctx.repeat(2), tau)
    for layer in range(2):
        single = wc.repair_select(terms[layer], norms[layer], ctx, tau)
        rows = slice(layer * wl.batch, (layer + 1) * wl.batch)
        for a, b in zip(stacked, single):
            assert torch.equal(a[rows], b)
