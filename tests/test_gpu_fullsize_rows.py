"""GPU parity of the §8(f) rows and the fused step at the benchmark's full
size (28 query / 4 KV heads, one sequence of 32768 tokens), in the calls the
benchmark makes, on sampled KV heads the oracle recomputes from the same
inputs:

  * the decode step with the new token's write fused in (bit for bit against
    write-then-decode, and against the oracle);
  * the Tier-B meter and the value-side terms;
  * block-level repair selection (contributions and the page-in lists);
  * the grouped-scale cache with 4 calibrated bypass pairs (write bit for bit,
    decode and grouped Tier B against the oracle)."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from oracle import quantizer as OQ
from tests._parity import assert_close, assert_sound, witness_step_up
from tests.test_gpu_repair import _check_selection

pytestmark = pytest.mark.gpu

LAYER, SEED = 11, 707


def _inputs():
    wl = W.config(2)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, LAYER, device="cuda")
    q = W.layer_queries(wl, LAYER, device="cuda")
    return wl, bt, sm, k, v, q


def assert_between(gpu, lo, hi, what):
    """A GPU result computed on its own write, whose witnesses may sit one fp16
    step above the oracle's: on or above the oracle's value for the oracle's
    witness (lo) and within tolerance of the oracle's value for every witness
    one step up (hi)."""
    assert_sound(gpu, lo, None, what)
    assert_close(np.maximum(gpu, hi), hi, f"{what} (witness one step up)")


def _oracle_head(wl, bt, k, v, h, scheme=OP.SCHEME_DITHER_INT8, pairs=None):
    """The oracle's reconstruction of KV head h of sequence 0 (all its tokens)."""
    m = 0 if pairs is None else pairs.shape[1]
    od = OP.Desc(num_q_heads=wl.n_q_heads, num_kv_heads=wl.n_kv_heads, num_pages=wl.num_pages, scheme=scheme,
                 seed=SEED, num_bypass_pairs=m)
    S = wl.ctx_lens[0]
    slots = OP.slots_of(od, bt[0], S)
    kr, vr = k[:S, h].cpu().numpy(), v[:S, h].cpu().numpy()
    excl = OQ.bypass_dims(pairs[h], 128, od.rope_layout) if m else ()
    kc, ks, khat = OP.quantize_rows(od, LAYER, h, kr, slots, 0, excl)
    vc, vs, vhat = OP.quantize_rows(od, LAYER, h, vr, slots, 1)
    w = OQ.witness(khat - kr.astype(np.float64), od.num_bands, od.rope_layout)
    vw = OQ.value_witness(vhat - vr.astype(np.float64), vr).astype(np.float64)
    return od, slots, kr, vr, kc, ks, khat, vc, vs, vhat, w, vw, excl


def test_fullsize_append_step():
    import paper_2607_28699_gb300 as wc
    from tests.test_gpu_fullsize import _check_cell
    wl, bt, sm, k, v, q = _inputs()
    gd = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=SEED)
    S = wl.ctx_lens[0]
    smd = torch.from_numpy(sm).cuda()
    base = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, LAYER, k[:S - 1].contiguous(), v[:S - 1].contiguous(), smd[:S - 1].contiguous(), base)
    a = wc.LayerCache(*(t.clone() for t in (base.k_codes, base.v_codes, base.k_scale, base.v_scale, base.k_witness)))
    kn, vn, sn = k[S - 1:].contiguous(), v[S - 1:].contiguous(), smd[S - 1:].contiguous()
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    btd = torch.from_numpy(bt).cuda()
    ws_a, ws_b = wc.Workspace(gd, 1, wl.max_pages), wc.Workspace(gd, 1, wl.max_pages)
    wc.kv_quantize_witness(gd, LAYER, kn, vn, sn, a)
    ra = wc.metered_decode_attention(gd, LAYER, q, btd, ctx, a, ws_a)
    rb = wc.metered_decode_attention_append(gd, LAYER, q, btd, ctx, base, ws_b, kn, vn, sn)
    torch.cuda.synchronize()
    assert wc.read_status(ws_a) == 0 and wc.read_status(ws_b) == 0
    for name in ("k_codes", "v_codes", "k_scale", "v_scale", "k_witness"):
        assert torch.equal(getattr(a, name), getattr(base, name)), name
    for x, y in zip(ra, rb):
        assert torch.equal(x, y)
    out, meter, raw = rb
    _check_cell(wl, LAYER, SEED, 0, 1, bt, k, v, q, base, out, meter, raw)


def test_fullsize_tier_b_and_value_side():
    import paper_2607_28699_gb300 as wc
    wl, bt, sm, k, v, q = _inputs()
    gd = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=SEED)
    cache = wc.LayerCache.empty(gd, value_witness=True)
    wc.kv_quantize_witness(gd, LAYER, k, v, torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, 1, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    btd = torch.from_numpy(bt).cuda()
    delta_loc = 1e-2 / (28 * 28)
    rb = wc.metered_decode_attention_tier_b(gd, LAYER, q, btd, ctx, cache, ws, delta_loc)
    rv = wc.metered_decode_attention_v(gd, LAYER, q, btd, ctx, cache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    h = 3
    od, slots, kr, vr, kc, ks, khat, vc, vs, vhat, w, vw, _ = _oracle_head(wl, bt, k, v, h)
    page, off = slots // 16, slots % 16
    g_vw = cache.v_witness[:, h].cpu().numpy()[page, off].astype(np.float64)
    vw16 = OQ.value_witness(vhat - vr.astype(np.float64), vr)
    vw_up = witness_step_up(vw16).astype(np.float64)
    assert np.all((g_vw == vw) | (g_vw == vw_up)) and np.all(g_vw >= vw)
    # the decode read the GPU's write, whose witnesses may be one fp16 step
    # above the oracle's: its results lie between the oracle's for the two ends
    w_up = witness_step_up(w).astype(np.float64)
    S = wl.ctx_lens[0]
    for g in range(wl.group):
        hq = h * wl.group + g
        qq = q[0, hq].cpu().numpy().astype(np.float64)
        pt = OM.softmax(OM.logits(qq, khat))
        u = OM.tier_b_bound(qq, ks.astype(np.float64), S, delta_loc)
        _, rb_ref, _ = OM.eform_meter(pt, u)
        assert_close(rb[4][0, hq].cpu().numpy(), rb_ref, f"meter_b_raw hq{hq}")
        assert_sound(rb[4][0, hq].cpu().numpy(), rb_ref, None, f"meter_b_raw hq{hq}")
        ends = []
        for ww, vv in ((w, vw), (w_up, vw_up)):
            meter_ref = min(1.0, OM.eform_meter(pt, OM.tier_a_bound(qq, ww, od.num_bands, od.rope_layout))[1])
            vt = OM.value_term(pt, vv[:, 0])
            ends.append((vt, np.max(vv[:, 1]), OM.output_bound(meter_ref, np.max(vv[:, 1]), vt)))
        assert_between(rv[3][0, hq].cpu().numpy(), ends[0][0], ends[1][0], f"value_term hq{hq}")
        assert ends[0][1] <= rv[4][0, hq].item() <= ends[1][1]
        assert_between(rv[5][0, hq].cpu().numpy(), ends[0][2], ends[1][2], f"out_bound hq{hq}")
        # the output bound holds against the exact output
        p = OM.softmax(OM.logits(qq, kr.astype(np.float64)))
        err = np.linalg.norm(OM.attend(p, vr.astype(np.float64)) - OM.attend(pt, vhat))
        assert err <= rv[5][0, hq].item()


def test_fullsize_repair_selection():
    import paper_2607_28699_gb300 as wc
    wl, bt, sm, k, v, q = _inputs()
    gd = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=SEED)
    cache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, LAYER, k, v, torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, 1, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    res = wc.metered_decode_attention_repair(gd, LAYER, q, torch.from_numpy(bt).cuda(), ctx, cache, ws)
    tau = 0.1                                               # the benchmark's gate
    keep_q, _, _ = wc.gate(res[2].reshape(-1), gd.group, tau)
    contrib, pages, n_rep, d_after = wc.repair_select(res[3], res[4], ctx, tau, keep_q=keep_q)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    h = 0
    od, slots, kr, vr, kc, ks, khat, vc, vs, vhat, w, vw, _ = _oracle_head(wl, bt, k, v, h)
    S = wl.ctx_lens[0]
    n = (S + 15) // 16
    keep = keep_q.cpu().numpy().astype(bool)
    w_up = witness_step_up(w).astype(np.float64)
    for g in range(wl.group):
        hq = h * wl.group + g
        qq = q[0, hq].cpu().numpy().astype(np.float64)
        pt = OM.softmax(OM.logits(qq, khat))
        ref_c = OM.page_contributions(pt, OM.tier_a_bound(qq, w, od.num_bands, od.rope_layout), np.arange(S) // 16, n)
        ref_up = OM.page_contributions(pt, OM.tier_a_bound(qq, w_up, od.num_bands, od.rope_layout),
                                       np.arange(S) // 16, n)
        gc = contrib[0, hq, :n].cpu().numpy()
        # between the oracle's contributions for the two witness ends (on the GPU's write)
        assert_close(np.minimum(gc, ref_c), ref_c, f"contrib hq{hq}", atol=1e-7)
        assert_close(np.maximum(gc, ref_up), ref_up, f"contrib hq{hq} (witness one step up)", atol=1e-7)
        if not keep[hq]:
            _check_selection(gc, pages[0, hq, :int(n_rep[0, hq])].cpu().numpy(), n, float(d_after[0, hq]), tau, ref_c)


def test_fullsize_grouped_with_calibrated_pairs():
    import paper_2607_28699_gb300 as wc
    wl, bt, sm, k, v, q = _inputs()
    gd = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=SEED,
                      scheme=wc.SCHEME_DITHER_INT8_G32)
    cache = wc.LayerCache.empty(gd, num_bypass_pairs=4)
    wc.select_bypass_pairs(k, 4, gd.rope_layout, pairs=cache.bypass_pairs)
    wc.kv_quantize_witness(gd, LAYER, k, v, torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, 1, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    delta_loc = 1e-2 / (28 * 28)
    out, meter, raw, mb, mb_raw = wc.metered_decode_attention_tier_b(gd, LAYER, q, torch.from_numpy(bt).cuda(), ctx,
                                                                     cache, ws, delta_loc)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    pairs = cache.bypass_pairs.cpu().numpy().astype(np.int64)
    h = 2
    od, slots, kr, vr, kc, ks, khat, vc, vs, vhat, w, vw, excl = _oracle_head(
        wl, bt, k, v, h, scheme=OP.SCHEME_DITHER_INT8_G32, pairs=pairs)
    page, off = slots // 16, slots % 16
    assert np.array_equal(cache.k_codes[:, h].cpu().numpy()[page, off], kc[:, OP.storage_order(128, 0)])
    assert np.array_equal(cache.v_codes[:, h].cpu().numpy()[page, off], vc[:, OP.storage_order(128, 1)])
    assert np.array_equal(cache.k_scale[:, h].cpu().numpy()[page, off].view(np.uint16), ks.view(np.uint16))
    assert np.array_equal(cache.v_scale[:, h].cpu().numpy()[page, off].view(np.uint16), vs.view(np.uint16))
    assert np.array_equal(cache.k_bypass[:, h].cpu().numpy()[page, off], kr[:, excl])
    g_w = cache.k_witness[:, h].cpu().numpy()[page, off].astype(np.float64)
    w_up = witness_step_up(w).astype(np.float64)
    assert np.all((g_w == w) | (g_w == w_up))
    S = wl.ctx_lens[0]
    for g in range(wl.group):
        hq = h * wl.group + g
        qq = q[0, hq].cpu().numpy().astype(np.float64)
        pt = OM.softmax(OM.logits(qq, khat))
        assert_close(out[0, hq].cpu().numpy(), OM.attend(pt, vhat), f"grouped out hq{hq}")
        lo = OM.eform_meter(pt, OM.tier_a_bound(qq, w, od.num_bands, od.rope_layout))[1]
        hi = OM.eform_meter(pt, OM.tier_a_bound(qq, w_up, od.num_bands, od.rope_layout))[1]
        assert_between(raw[0, hq].cpu().numpy(), lo, hi, f"grouped meter_raw hq{hq}")
        u = OM.tier_b_bound_grouped(qq, ks, 32, excl, S, delta_loc)
        assert_close(mb_raw[0, hq].cpu().numpy(), OM.eform_meter(pt, u)[1], f"grouped meter_b_raw hq{hq}")
        assert_sound(mb_raw[0, hq].cpu().numpy(), OM.eform_meter(pt, u)[1], None, f"grouped meter_b_raw hq{hq}")
