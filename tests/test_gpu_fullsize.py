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
above the oracle's (never below), outputs and meters within 1e-3 relative /
1e-5 absolute, and gate decisions bit for bit on the same fp32 meters."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from oracle import quantizer as OQ
from tests._parity import assert_close

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
    res_out, res_raw = [], []
    for g in range(G):
        hq = h * G + g
        qq = q[b, hq].cpu().numpy().astype(np.float64)
        pt = OM.softmax(OM.logits(qq, khat))
        c = OM.tier_a_bound(qq, w, od.num_bands, od.rope_layout)
        _, r, _ = OM.eform_meter(pt, c)
        res_out.append(OM.attend(pt, vhat))
        res_raw.append(r)
        # soundness at full size: the meter bounds the true TV
        p = OM.softmax(OM.logits(qq, kr.astype(np.float64)))
        assert OM.total_variation(p, pt) <= r * (1 + 1e-12)
    sl = slice(h * G, (h + 1) * G)
    assert_close(out[b, sl].cpu().numpy(), np.stack(res_out), f"out b{b} h{h}")
    assert_close(raw[b, sl].cpu().numpy(), np.array(res_raw), f"meter_raw b{b} h{h}")
    assert_close(meter[b, sl].cpu().numpy(), np.minimum(1.0, np.array(res_raw)), f"meter b{b} h{h}")


def test_fullsize_28L_S32768():
    wl = W.config(2)
    layer, seed = 13, 101
    gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
    _check_cell(wl, layer, seed, 0, 2, bt, k, v, q, cache, out, meter, raw)


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
    _check_cell(wl, layer, seed, 0, 1, bt, k, v, q, cache, out, meter, raw)


def test_fullsize_fp8_batch32_gated():
    import paper_2607_28699_gb300 as wc
    wl = W.config(5)
    layer, seed = 5, 404
    gd, bt, sm, k, v, q, cache, out, meter, raw = _gpu_layer(wl, layer, seed)
    for b, h in [(3, 0), (20, 2), (31, 3)]:
        _check_cell(wl, layer, seed, b, h, bt, k, v, q, cache, out, meter, raw)
    flat = raw.reshape(-1)
    for tau in wl.taus:
        keep_q, keep_kv, kept = wc.gate(flat, gd.group, tau)
        oq, okv, nq, nkv = OM.gate(flat.cpu().numpy(), tau, gd.group)
        assert np.array_equal(keep_q.cpu().numpy().astype(bool), oq)
        assert np.array_equal(keep_kv.cpu().numpy().astype(bool), okv)
        assert kept.cpu().tolist() == [nq, nkv]
