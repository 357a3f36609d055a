"""GPU parity of the grouped-scale cache with the fixed-channel outlier-pair
bypass (§6.2.3 "Storage side", §6.2.5 "Fixed-channel outlier bypass"): the write
kernel's codes (in storage order), group scales and exact bypassed values bit
for bit against the oracle, its witness at most one fp16 step above; the
decode's output, meter and grouped Tier-B meter against the oracle on
ragged, paged contexts with m = 0, 2, 4 and 16 bypassed pairs in both RoPE
layouts; the pair calibration; an out-of-range pair index reported, not
trapped."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from oracle import quantizer as Q
from tests._parity import assert_close, assert_sound, descs, gpu_cache_to_numpy, make_inputs, numpy_cache_to_gpu

pytestmark = pytest.mark.gpu


def _pairs(m, hkv, seed):
    rng = np.random.default_rng(seed)
    return np.stack([np.sort(rng.choice(64, m, replace=False)) for _ in range(hkv)]).astype(np.int64)


def _massive(k, pairs, layout, factor=30.0):
    """Keys with the bypass pairs made massive (the massive-activation effect)."""
    k = k.copy()
    for h in range(k.shape[1]):
        if pairs.shape[1]:
            dims = Q.bypass_dims(pairs[h], 128, layout)
            k[:, h, dims] = (k[:, h, dims].astype(np.float32) * factor).astype(np.float16)
    return k


def _write_both(wl, layer, m, layout, seed):
    import paper_2607_28699_gb300 as wc
    bt, sm, k, v, q = make_inputs(wl, layer)
    pairs = _pairs(m, wl.n_kv_heads, seed)
    k = _massive(k.numpy(), pairs, layout)
    v = v.numpy()
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, OP.SCHEME_DITHER_INT8_G32, 8, layout, seed,
                   num_bypass_pairs=m)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k, v, sm, ocache, bypass_pairs=pairs if m else None)
    gcache = wc.LayerCache.empty(gd, num_bypass_pairs=m)
    if m:
        gcache.bypass_pairs.copy_(torch.from_numpy(pairs.astype(np.int32)))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    wc.kv_quantize_witness(gd, layer, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                           torch.from_numpy(sm).cuda(), gcache, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return bt, k, v, q, od, gd, ocache, gcache


def _check_write(ocache, gcache):
    g = gpu_cache_to_numpy(gcache)
    for name in ("k_codes", "v_codes", "k_scale", "v_scale") + (("k_bypass",) if "k_bypass" in g else ()):
        assert np.array_equal(g[name].view(np.uint8), ocache[name].view(np.uint8)), name
    ow = ocache["k_witness"].astype(np.float64)
    gw = g["k_witness"].astype(np.float64)
    up = (ocache["k_witness"].view(np.uint16) + 1).view(np.float16).astype(np.float64)
    assert np.all(gw >= ow) and np.all((gw == ow) | (gw == up))


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
@pytest.mark.parametrize("m", [0, 2, 4, 16])
def test_grouped_write_matches_oracle(m, layout):
    wl = W.Workload("gw", 1, 8, 2, [700, 33, 5], shuffle_pages=True, seed=21 + m)
    *_, ocache, gcache = _write_both(wl, 1, m, layout, 3 + m)
    _check_write(ocache, gcache)


@pytest.mark.parametrize("n_tok", [1, 3, 15])
def test_grouped_write_small_batches(n_tok):
    """Fewer than 16 tokens take the kernel's one-index grid."""
    wl = W.Workload("gs", 1, 8, 4, [n_tok], shuffle_pages=True, seed=31)
    *_, ocache, gcache = _write_both(wl, 0, 4, Q.ROPE_HALF, 7)
    _check_write(ocache, gcache)


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
@pytest.mark.parametrize("m", [0, 2, 4, 16])
def test_grouped_decode_matches_oracle(m, layout):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("gd", 1, 28, 4, [4100, 77, 1, 1600, 16], shuffle_pages=True, seed=41 + m)
    layer = 2
    bt, k, v, q, od, gd, ocache, _ = _write_both(wl, layer, m, layout, 11 + m)
    gcache = numpy_cache_to_gpu(ocache, gd)     # identical stored inputs on both sides
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    delta = 1e-4
    out, meter, raw = wc.metered_decode_attention(gd, layer, qd, btd, ctx, gcache, ws)
    res_b = wc.metered_decode_attention_tier_b(gd, layer, qd, btd, ctx, gcache, ws, delta)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    assert torch.equal(out, res_b[0]) and torch.equal(raw, res_b[2])    # Tier B leaves the rest alone
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    ref = {n: [] for n in ("out", "meter_raw", "meter_b_raw", "tv")}
    for b, S in enumerate(wl.ctx_lens):
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k[offs[b]:offs[b] + S],
                               v[offs[b]:offs[b] + S], delta_loc=delta)
        for n in ref:
            ref[n].append(r[n])
    ref = {n: np.stack(x) for n, x in ref.items()}
    assert_close(out.cpu().numpy(), ref["out"], f"out m={m}")
    assert_close(raw.cpu().numpy(), ref["meter_raw"], f"meter_raw m={m}")
    assert_close(res_b[4].cpu().numpy(), ref["meter_b_raw"], f"meter_b_raw m={m}")
    assert_sound(raw.cpu().numpy(), ref["meter_raw"], ref["tv"], f"meter_raw m={m}")
    assert_sound(res_b[4].cpu().numpy(), ref["meter_b_raw"], None, f"meter_b_raw m={m}")


@pytest.mark.parametrize("ctx_lens", [[0, 1, 16, 17, 40, 0, 33, 5] * 25, [3000, 1, 0, 16, 2049, 17, 0, 700],
                                      [(37 * i) % 41 for i in range(500)]])
def test_grouped_decode_flattened_plan_batches(ctx_lens):
    """A batch runs the grouped decode under the flattened split plan (6 page
    streams per CTA, shares cut at sequence boundaries): every sequence against
    the oracle, with and without Tier B; empty sequences give out = 0, meter 0."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("gf", 1, 28, 4, ctx_lens, shuffle_pages=True, seed=61)
    layer, m = 1, 4
    bt, k, v, q, od, gd, ocache, _ = _write_both(wl, layer, m, Q.ROPE_HALF, 17)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    delta = 1e-4
    out, meter, raw = wc.metered_decode_attention(gd, layer, qd, btd, ctx, gcache, ws)
    res_b = wc.metered_decode_attention_tier_b(gd, layer, qd, btd, ctx, gcache, ws, delta)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, raw, raw_b = out.cpu().numpy(), raw.cpu().numpy(), res_b[4].cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(ctx_lens)[:-1]])
    for b, S in enumerate(ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(raw[b] == 0) and np.all(raw_b[b] == 0)
            continue
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k[offs[b]:offs[b] + S],
                               v[offs[b]:offs[b] + S], delta_loc=delta)
        assert_close(out[b], r["out"], f"out[{b}]")
        assert_close(raw[b], r["meter_raw"], f"meter_raw[{b}]")
        assert_close(raw_b[b], r["meter_b_raw"], f"meter_b_raw[{b}]")
        assert_sound(raw[b], r["meter_raw"], r["tv"], f"meter_raw[{b}]")
        assert_sound(raw_b[b], r["meter_b_raw"], None, f"meter_b_raw[{b}]")


def test_grouped_bypass_lowers_the_meter_on_massive_pairs():
    """Table "amax" on the GPU path: with massive pairs, the grouped cache
    that bypasses them (and leaves them out of the amax) meters far lower."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("ga", 1, 8, 2, [2048], shuffle_pages=True, seed=51)
    bt, sm, k, v, q = make_inputs(wl, 0)
    pairs = _pairs(4, 2, 5)
    k = _massive(k.numpy(), pairs, Q.ROPE_HALF, factor=60.0)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    meters = {}
    for m in (0, 4):
        gd = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=wc.SCHEME_DITHER_INT8_G32,
                          seed=3)
        cache = wc.LayerCache.empty(gd, num_bypass_pairs=m)
        if m:
            cache.bypass_pairs.copy_(torch.from_numpy(pairs.astype(np.int32)))
        wc.kv_quantize_witness(gd, 0, torch.from_numpy(k).cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
        ws = wc.Workspace(gd, 1, wl.max_pages)
        res = wc.metered_decode_attention_tier_b(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx, cache, ws, 1e-4)
        meters[m] = float(res[4].median())
    assert meters[4] < meters[0] / 10, meters


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
def test_pair_calibration_matches_oracle(layout):
    import paper_2607_28699_gb300 as wc
    rng = np.random.default_rng(61)
    n, hkv = 500, 4
    k = (rng.standard_normal((n, hkv, 128)) * np.exp(rng.normal(0, 0.5, (1, hkv, 128)))).astype(np.float16)
    pairs = _pairs(8, hkv, 62)
    k = _massive(k, pairs, layout, factor=20.0)
    got = wc.select_bypass_pairs(torch.from_numpy(k).cuda(), 8, layout).cpu().numpy()
    for h in range(hkv):
        assert np.array_equal(got[h], Q.select_bypass_pairs(k[:, h], 8, layout))
        assert np.array_equal(got[h], pairs[h])
    # without a planted structure: the chosen energies are a top set (fp32 sums)
    k2 = rng.standard_normal((n, hkv, 128)).astype(np.float16)
    got2 = wc.select_bypass_pairs(torch.from_numpy(k2).cuda(), 5, layout).cpu().numpy()
    for h in range(hkv):
        x = k2[:, h].astype(np.float64)
        dims = Q.bypass_dims(np.arange(64), 128, layout).reshape(64, 2)
        e = np.sum(x[:, dims[:, 0]] ** 2 + x[:, dims[:, 1]] ** 2, axis=0)
        chosen, rest = e[got2[h]], np.delete(e, got2[h])
        assert np.all(np.diff(got2[h]) > 0) and chosen.min() >= rest.max() * (1 - 1e-5)


def test_out_of_range_pair_is_reported_and_ignored():
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("gp", 1, 8, 2, [100], shuffle_pages=False, seed=71)
    bt, sm, k, v, q = make_inputs(wl, 0)
    gd = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=wc.SCHEME_DITHER_INT8_G32)
    cache = wc.LayerCache.empty(gd, num_bypass_pairs=2)
    cache.bypass_pairs.copy_(torch.tensor([[3, 64], [-1, 9]], dtype=torch.int32))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & wc.DEV_BAD_PAIR
    assert torch.all(cache.k_bypass[..., 2:4][:, 0] == 0) and torch.all(cache.k_bypass[..., 0:2][:, 1] == 0)
    ws = wc.Workspace(gd, 1, wl.max_pages)
    out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(),
                                                  torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda"),
                                                  cache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) & wc.DEV_BAD_PAIR
    assert torch.isfinite(out).all() and torch.isfinite(raw).all()


def test_repeated_pair_is_ignored_like_an_out_of_range_one():
    """A pair listed twice counts once: its second occurrence is reported and
    stores zeros, exactly like an out-of-range index in its place."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("gr", 1, 8, 2, [300, 20], shuffle_pages=True, seed=73)
    bt, sm, k, v, q = make_inputs(wl, 0)
    k = _massive(k.numpy(), np.array([[5, 11], [7, 8]]), Q.ROPE_HALF)
    gd = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=wc.SCHEME_DITHER_INT8_G32)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    res = []
    for pairs in ([[5, 11, 5], [7, 8, 8]], [[5, 11, -1], [7, 8, 64]]):
        for n_split in (None, 3):   # the per-head grid (all tokens) and the one-index grid (3 tokens at a time)
            cache = wc.LayerCache.empty(gd, num_bypass_pairs=3)
            cache.bypass_pairs.copy_(torch.tensor(pairs, dtype=torch.int32))
            status = torch.zeros(1, dtype=torch.int32, device="cuda")
            kd, vd, sd = torch.from_numpy(k).cuda(), v.cuda(), torch.from_numpy(sm).cuda()
            chunks = [slice(0, len(sm))] if n_split is None else [slice(i, i + n_split) for i in range(0, len(sm), n_split)]
            for ch in chunks:
                wc.kv_quantize_witness(gd, 0, kd[ch].contiguous(), vd[ch].contiguous(), sd[ch].contiguous(), cache,
                                       dev_status=status)
            ws = wc.Workspace(gd, wl.batch, wl.max_pages)
            out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx, cache, ws)
            torch.cuda.synchronize()
            assert int(status.item()) & wc.DEV_BAD_PAIR and wc.read_status(ws) & wc.DEV_BAD_PAIR
            res.append((cache.k_codes.clone(), cache.k_bypass.clone(), out, raw))
    for other in res[1:]:
        for a, b in zip(res[0], other):
            assert torch.equal(a, b)
