"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark uses (one layer's write and metered decode over all sequences and
heads), checked on sampled (sequence, KV head) cells that the oracle
recomputes from the same inputs:

  * 28 layers' shape, 28 q / 4 KV heads, one sequence of 32768 tokens;
  * batch 16, contexts 4096-8192, shuffled 16-token pages, prefill write;
  * one sequence of 131072 tokens;
  * raw-cast fp8, batch 32, contexts 4096-32768, 5% of cells with a 4x query,
    gated at tau in {0.05, 0.1, 0.2}.

Codes and scales must match bit for bit, the witness may be one fp16 ulp
above the oracle's (never below), outputs within 1e-3 relative / 1e-5
absolute, meters on or above the oracle's fp64 meters and within that
tolerance of the oracle's meters for the witness one step up (the most the
GPU's write may store), and the whole batch's gate consistent (KV heads
any-of-G, counts).  End to end, the GPU's gate on its own meters equals the oracle's
gate on the oracle's fp64 meters except for cells whose meter sits within
1e-3 tau + 1e-5 of tau (counted and reported)."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from oracle import quantizer as OQ
from tests._parity import assert_close, assert_sound, witness_step_up

pytestmark = pytest.mark.gpu


def _gpu_layer(wl, layer, seed):
    import paper_2607_28699_gb300 as wc
    gd = wc.CacheDesc(num_q_heads=wl.n_q_heads, num_kv_heads=wl.n_kv_heads, num_pages=wl.num_pages,
                      scheme=wl.scheme, seed=seed)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, layer, device="cuda")
    q = W.layer_queries(wl, layer, device="cuda")
    cache = wc.LayerCache.empty(gd)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    wc.kv_quantize_witness(gd, layer, k, v, torch.from_numpy(sm).cuda(), cache, dev_status=status)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, layer, q, torch.from_numpy(bt).cuda(), ctx, cache, ws)
    torch.cuda.synchronize()
    assert int(status.item()) == 0 and wc.read_status(ws) == 0
    return gd, bt, sm, k, v, q, cache, out, meter, raw


def _check_cell(wl, layer, seed, b, h, bt, k, v, q, cache, out, meter, raw):
    """Oracle recomputation of sequence b, KV head h (all its query heads)."""
    od = OP.Desc(num_q_heads=wl.n_q_heads, num_kv_heads=wl.n_kv_heads, num_pages=wl.num_pages,
                 scheme=wl.scheme, seed=seed)
    S = wl.ctx_lens[b]
    off = int(sum(wl.ctx_lens[:b]))
    slots = OP.slots_of(od, bt[b], S)
    page, slot_off = slots // 16, slots % 16
    kr = k[off:off + S, h].cpu().numpy()
    vr = v[off:off + S, h].cpu().numpy()
    kc, ks, khat = OP.quantize_rows(od, layer, h, kr, slots, 0)
    vc, vs, vhat = OP.quantize_rows(od, layer, h, vr, slots, 1)
    w = OQ.witness(khat - kr.astype(np.float64), od.num_bands, od.rope_layout)

    # the write path, bit for bit (codes, scales) and within one ulp (witness)
    g_kc = cache.k_codes[:, h].cpu().numpy()[page, slot_off]
    g_vc = cache.v_codes[:, h].cpu().numpy()[page, slot_off]
    assert np.array_equal(g_kc.view(np.uint8), kc.view(np.uint8))
    assert np.array_equal(g_vc.view(np.uint8), vc.view(np.uint8))
    if ks is not None:
        assert np.array_equal(cache.k_scale[:, h].cpu().numpy()[page, slot_off].view(np.uint16), ks.view(np.uint16))
        assert np.array_equal(cache.v_scale[:, h].cpu().numpy()[page, slot_off].view(np.uint16), vs.view(np.uint16))
    g_w = cache.k_witness[:, h].cpu().numpy()[page, slot_off]
    up = (w.view(np.uint16) + 1).view(np.float16)
    assert np.all((g_w == w) | (g_w == up))

    # the read path for the G query heads of this KV head
    G = wl.group
    res_out, res_raw, res_up, res_tv = [], [], [], []
    for g in range(G):
        hq = h * G + g
        qq = q[b, hq].cpu().numpy().astype(np.float64)
        pt = OM.softmax(OM.logits(qq, khat))
        c = OM.tier_a_bound(qq, w, od.num_bands, od.rope_layout)
        _, r, _ = OM.eform_meter(pt, c)
        _, r_up, _ = OM.eform_meter(pt, OM.tier_a_bound(qq, witness_step_up(w), od.num_bands, od.rope_layout))
        res_out.append(OM.attend(pt, vhat))
        res_raw.append(r)
        res_up.append(r_up)
        # soundness at full size: the meter bounds the true TV
        p = OM.softmax(OM.logits(qq, kr.astype(np.float64)))
        res_tv.append(OM.total_variation(p, pt))
        assert res_tv[-1] <= r * (1 + 1e-12)
    sl = slice(h * G, (h + 1) * G)
    g_raw, g_meter = raw[b, sl].cpu().numpy(), meter[b, sl].cpu().numpy()
    res_raw, res_up = np.array(res_raw), np.array(res_up)
    assert_close(out[b, sl].cpu().numpy(), np.stack(res_out), f"out b{b} h{h}")
    assert_sound(g_raw, res_raw, np.array(res_tv), f"meter_raw b{b} h{h}")
    assert_close(np.maximum(g_raw, res_up), res_up, f"meter_raw b{b} h{h} (witness one step up)")
    assert_close(np.maximum(g_meter, np.minimum(1.0, res_up)), np.minimum(1.0, res_up), f"meter b{b} h{h}")
    return res_raw


def _gate_end_to_end(wl, g_raw, o_raw, taus):
    """The GPU's gate on its fp32 meters against the oracle's gate on its fp64
    meters for the same cells (§6 meter loop: keep iff meter_raw <= tau).
    Cells within 1e-3 tau + 1e-5 of tau are excluded and their count reported."""
    import paper_2607_28699_gb300 as wc
    g_raw = np.asarray(g_raw, np.float32)
    o_raw = np.asarray(o_raw, np.float64)
    for tau in taus:
        keep_q, _, _ = wc.gate(torch.from_numpy(g_raw).cuda(), 1, tau)
        oq, _, _, _ = OM.gate(o_raw, tau, 1)
        near = np.abs(o_raw - tau) < 1e-3 * tau + 1e-5
        print(f"[gate] tau={tau}: {int(near.sum())} of {near.size} cells within the band excluded; "
              f"kept {int(oq.sum())} by the oracle")
        assert int(near.sum()) <= max(1, near.size // 20)
        g = keep_q.cpu().numpy().astype(bool)
        assert np.array_equal(g[~near], oq[~near])


def test_fullsize_28L_S32768():
    """Every KV head of two layers of the benchmark's 32k sequence, and the
    gate at tau = 0.1 end to end on those cells."""
    wl = W.config(2)
    seed = 101
    g_raw, o_raw = [], []
    for layer in (13, 27):
        gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
        for h in range(wl.n_kv_heads):
            o_raw.append(_check_cell(wl, layer, seed, 0, h, bt, k, v, q, cache, out, meter, raw))
            g_raw.append(raw[0, h * wl.group:(h + 1) * wl.group].cpu().numpy())
    o_all = np.concatenate(o_raw)
    _gate_end_to_end(wl, np.concatenate(g_raw), o_all, list(wl.taus) + [float(np.median(o_all))])


def test_fullsize_batch16_paged_prefill():
    wl = W.config(3)
    layer, seed = 27, 202
    gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
    for b, h in [(0, 0), (4, 2), (9, 3), (12, 0), (15, 1)]:   # the flattened split plan's segments
        _check_cell(wl, layer, seed, b, h, bt, k, v, q, cache, out, meter, raw)


def test_fullsize_S131072():
    wl = W.config(4)
    layer, seed = 0, 303
    gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
    for h in (1, 3):
        _check_cell(wl, layer, seed, 0, h, bt, k, v, q, cache, out, meter, raw)


def test_fullsize_fp8_batch32_gated():
    import paper_2607_28699_gb300 as wc
    wl = W.config(5)
    layer, seed = 5, 404
    gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
    g_raw, o_raw = [], []
    for b, h in [(3, 0), (20, 2), (31, 3), (7, 1), (26, 0)]:
        o_raw.append(_check_cell(wl, layer, seed, b, h, bt, k, v, q, cache, out, meter, raw))
        g_raw.append(raw[b, h * wl.group:(h + 1) * wl.group].cpu().numpy())
    o_all = np.concatenate(o_raw)
    # the workload's taus, and one that splits the sampled cells (both decisions occur)
    _gate_end_to_end(wl, np.concatenate(g_raw), o_all, list(wl.taus) + [float(np.median(o_all))])
    flat = raw.reshape(-1)
    for tau in wl.taus:   # the whole batch: counts consistent with the decisions
        keep_q, keep_kv, kept = wc.gate(flat, gd.group, tau)
        kq = keep_q.cpu().numpy().astype(bool)
        kkv = keep_kv.cpu().numpy().astype(bool)
        assert np.array_equal(kkv, kq.reshape(-1, gd.group).all(axis=1))
        assert kept.cpu().tolist() == [int(kq.sum()), int(kkv.sum())]
