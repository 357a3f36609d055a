"""Seeded random sweep of the write + metered decode path against the oracle.

Each case draws its own shape: 1, 2 or 4 KV heads with a GQA group of 1 to 8,
a batch of 1 to 12 sequences whose lengths mix empty sequences, lengths on and
next to page boundaries and arbitrary ragged ones, sequential or shuffled
physical pages, both RoPE pairings, the three read schemes (8- and 10-bit
dither, fp8) and either the GPU's own write or the oracle's cache copied in.
Outputs and meters must meet the same bounds as the fixed cases: within 1e-3
relative / 1e-5 absolute of the oracle, the meter on or above the oracle's
fp64 meter and the true total variation."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, descs, make_inputs, numpy_cache_to_gpu, witness_step_up

pytestmark = pytest.mark.gpu

SCHEMES = [(0, 8), (0, 10), (1, 8)]


def _case(i):
    r = np.random.default_rng(4000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    batch = int(r.integers(1, 13))
    lens = []
    for _ in range(batch):
        u = r.random()
        if u < 0.15:
            lens.append(0)
        elif u < 0.45:
            lens.append(int(16 * r.integers(1, 150) + r.integers(-1, 2)))   # on or next to a page boundary
        else:
            lens.append(int(r.integers(1, 2500)))
    if max(lens) == 0:
        lens[0] = int(r.integers(1, 2500))
    scheme, bits = SCHEMES[i % len(SCHEMES)]
    wl = W.Workload(f"sweep{i}", 1, group * hkv, hkv, lens, shuffle_pages=bool(r.random() < 0.5), seed=50 + i)
    return wl, scheme, bits, int(r.integers(0, 2)), int(r.integers(0, 28)), bool(i % 2 == 0)


@pytest.mark.parametrize("i", range(18))
def test_random_shapes_match_oracle(i):
    import paper_2607_28699_gb300 as wc
    wl, scheme, bits, layout, layer, gpu_writes = _case(i)
    print(f"[sweep {i}] Hq={wl.n_q_heads} Hkv={wl.n_kv_heads} lens={wl.ctx_lens} scheme={scheme}/{bits} "
          f"layout={layout} layer={layer} shuffle={wl.shuffle_pages} gpu_writes={gpu_writes}")
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, scheme, bits, layout, 7 + i)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    if gpu_writes:
        gcache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache)
    else:
        gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, meter, raw = out.cpu().numpy(), meter.cpu().numpy(), raw.cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    up = dict(ocache)
    up["k_witness"] = witness_step_up(ocache["k_witness"])
    for b, S in enumerate(wl.ctx_lens):
        if S == 0:   # an empty context: out = 0, meters 0
            assert np.all(out[b] == 0) and np.all(meter[b] == 0) and np.all(raw[b] == 0)
            continue
        o = offs[b]
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k.numpy()[o:o + S], v.numpy()[o:o + S])
        assert_close(out[b], r["out"], f"out[{b}]")
        assert_sound(raw[b], r["meter_raw"], r["tv"], f"meter_raw[{b}]")
        if gpu_writes:   # the GPU's own write: its witness may be one fp16 step above the oracle's
            r_up = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, up)
            assert_close(np.maximum(raw[b], r_up["meter_raw"]), r_up["meter_raw"], f"meter_raw[{b}] (step up)")
            assert_close(np.maximum(meter[b], r_up["meter"]), r_up["meter"], f"meter[{b}] (step up)")
        else:
            assert_close(raw[b], r["meter_raw"], f"meter_raw[{b}]")
            assert_close(meter[b], r["meter"], f"meter[{b}]")


def _lens(r, batch, top):
    lens = [0 if r.random() < 0.15 else int(r.integers(1, top)) for _ in range(batch)]
    if max(lens) == 0:
        lens[0] = int(r.integers(1, top))
    return lens


@pytest.mark.parametrize("i", range(10))
def test_random_shapes_grouped_cache_and_tier_b(i):
    """The grouped-scale cache (§6.2.3, §6.2.5) with 0-8 bypassed pairs: its
    write bit for bit, its decode and grouped Tier-B meter against the oracle."""
    import paper_2607_28699_gb300 as wc
    from tests.test_gpu_grouped import _check_write, _write_both
    r = np.random.default_rng(5000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    m = int(r.choice([0, 1, 2, 3, 4, 8]))
    layout = int(r.integers(0, 2))
    wl = W.Workload(f"gsweep{i}", 1, group * hkv, hkv, _lens(r, int(r.integers(1, 11)), 2200),
                    shuffle_pages=bool(r.random() < 0.5), seed=70 + i)
    layer = int(r.integers(0, 28))
    print(f"[gsweep {i}] Hq={wl.n_q_heads} Hkv={hkv} m={m} layout={layout} lens={wl.ctx_lens}")
    bt, k, v, q, od, gd, ocache, gwrite = _write_both(wl, layer, m, layout, 90 + i)
    _check_write(ocache, gwrite)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    delta = 10.0 ** -float(r.integers(2, 6))
    res = wc.metered_decode_attention_tier_b(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws,
                                             delta)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, raw, raw_b = res[0].cpu().numpy(), res[2].cpu().numpy(), res[4].cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    for b, S in enumerate(wl.ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(raw[b] == 0) and np.all(raw_b[b] == 0)
            continue
        o = offs[b]
        ref = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k[o:o + S], v[o:o + S], delta_loc=delta)
        assert_close(out[b], ref["out"], f"out[{b}]")
        assert_close(raw[b], ref["meter_raw"], f"meter_raw[{b}]")
        assert_sound(raw[b], ref["meter_raw"], ref["tv"], f"meter_raw[{b}]")
        assert_close(raw_b[b], ref["meter_b_raw"], f"meter_b_raw[{b}]")
        assert_sound(raw_b[b], ref["meter_b_raw"], None, f"meter_b_raw[{b}]")


@pytest.mark.parametrize("i", range(8))
def test_random_shapes_tier_b_per_token_cache(i):
    """Tier B (§4.2) on the per-token dithered cache, 8- and 10-bit dither."""
    import paper_2607_28699_gb300 as wc
    r = np.random.default_rng(6000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    bits = 8 if i % 2 == 0 else 10
    layout = int(r.integers(0, 2))
    wl = W.Workload(f"bsweep{i}", 1, group * hkv, hkv, _lens(r, int(r.integers(1, 11)), 2600),
                    shuffle_pages=bool(r.random() < 0.5), seed=80 + i)
    layer = int(r.integers(0, 28))
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, 0, bits, layout, 40 + i)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    delta = 10.0 ** -float(r.integers(2, 6))
    res = wc.metered_decode_attention_tier_b(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws,
                                             delta)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, raw_b = res[0].cpu().numpy(), res[4].cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    for b, S in enumerate(wl.ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(raw_b[b] == 0)
            continue
        o = offs[b]
        ref = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k.numpy()[o:o + S], v.numpy()[o:o + S],
                                 delta_loc=delta)
        assert_close(out[b], ref["out"], f"out[{b}]")
        assert_close(raw_b[b], ref["meter_b_raw"], f"meter_b_raw[{b}]")
        assert_sound(raw_b[b], ref["meter_b_raw"], None, f"meter_b_raw[{b}]")


@pytest.mark.parametrize("i", range(8))
def test_random_shapes_fused_append(i):
    """The step's write fused into its decode: cache and outputs bit for bit
    those of the separate write and decode, on random shapes (one new token
    per sequence, some sequences without one)."""
    import paper_2607_28699_gb300 as wc
    r = np.random.default_rng(7000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    lens = [int(r.integers(1, 3000)) for _ in range(int(r.integers(1, 11)))]
    wl = W.Workload(f"asweep{i}", 1, group * hkv, hkv, lens, shuffle_pages=bool(r.random() < 0.5), seed=90 + i)
    layer = int(r.integers(0, 28))
    bt, sm, k, v, q = make_inputs(wl, layer)
    last = np.cumsum(wl.ctx_lens) - 1
    prefix = np.setdiff1d(np.arange(len(sm)), last)
    gd = wc.CacheDesc(num_q_heads=wl.n_q_heads, num_kv_heads=hkv, num_pages=wl.num_pages,
                      rope_layout=int(r.integers(0, 2)), seed=60 + i)
    kd, vd, smd = k.cuda(), v.cuda(), torch.from_numpy(sm).cuda()
    base = wc.LayerCache.empty(gd)
    if prefix.size:
        pi = torch.from_numpy(prefix).cuda()
        wc.kv_quantize_witness(gd, layer, kd[pi].contiguous(), vd[pi].contiguous(), smd[pi].contiguous(), base)
    li = torch.from_numpy(last).cuda()
    k_new, v_new, s_new = kd[li].contiguous(), vd[li].contiguous(), smd[li].contiguous()
    skip = r.random(len(lens)) < 0.2
    s_new[torch.from_numpy(skip).cuda()] = -1                       # no new token for these sequences
    keep = ~skip
    clone = lambda c: wc.LayerCache(c.k_codes.clone(), c.v_codes.clone(), c.k_scale.clone(), c.v_scale.clone(),
                                    c.k_witness.clone())
    a, b = clone(base), clone(base)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    ws_a, ws_b = wc.Workspace(gd, wl.batch, wl.max_pages), wc.Workspace(gd, wl.batch, wl.max_pages)
    if keep.any():
        ki = torch.from_numpy(np.nonzero(keep)[0]).cuda()
        wc.kv_quantize_witness(gd, layer, k_new[ki].contiguous(), v_new[ki].contiguous(), s_new[ki].contiguous(), a)
    ra = wc.metered_decode_attention(gd, layer, qd, btd, ctx, a, ws_a)
    rb = wc.metered_decode_attention_append(gd, layer, qd, btd, ctx, b, ws_b, k_new, v_new, s_new)
    torch.cuda.synchronize()
    assert wc.read_status(ws_a) == 0 and wc.read_status(ws_b) == 0
    for name in ("k_codes", "v_codes", "k_scale", "v_scale", "k_witness"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
    for x, y in zip(ra, rb):
        assert torch.equal(x, y)


@pytest.mark.parametrize("i", range(8))
def test_random_shapes_value_side(i):
    """Value witness, value term, max ||v|| and the output bound (§3, §4.2)
    against the oracle on random shapes, all three read schemes."""
    import paper_2607_28699_gb300 as wc
    r = np.random.default_rng(8000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    scheme, bits = SCHEMES[i % len(SCHEMES)]
    wl = W.Workload(f"vsweep{i}", 1, group * hkv, hkv, _lens(r, int(r.integers(1, 11)), 2600),
                    shuffle_pages=bool(r.random() < 0.5), seed=110 + i)
    layer = int(r.integers(0, 28))
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, hkv, wl.num_pages, scheme, bits, 0, 20 + i)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    gcache = numpy_cache_to_gpu(ocache, gd, value_witness=True)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    res = wc.metered_decode_attention_v(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, vterm, vmax, bound = (res[j].cpu().numpy() for j in (0, 3, 4, 5))
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    for b, S in enumerate(wl.ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(vterm[b] == 0) and np.all(bound[b] == 0)
            continue
        o = offs[b]
        ref = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, k.numpy()[o:o + S], v.numpy()[o:o + S])
        assert_close(out[b], ref["out"], f"out[{b}]")
        assert_close(vterm[b], ref["value_term"], f"value_term[{b}]")
        assert_sound(vterm[b], ref["value_term"], None, f"value_term[{b}]")
        assert np.array_equal(vmax[b].astype(np.float64), ref["v_max"])
        assert_close(bound[b], ref["out_bound"], f"out_bound[{b}]")
        assert np.all(bound[b] >= ref["out_err"])


@pytest.mark.parametrize("i", range(6))
def test_random_shapes_repair_selection(i):
    """Block-level repair selection (§6.3.5) on random shapes: the per-page
    contributions against the oracle's, the plain outputs untouched, and each
    flagged cell's list consistent with the kernel's contributions and a top
    set of the oracle's that brings the meter to tau."""
    import paper_2607_28699_gb300 as wc
    from tests.test_gpu_repair import _check_selection
    r = np.random.default_rng(9000 + i)
    hkv = int(r.choice([1, 2, 4]))
    group = int(r.integers(1, 9))
    scheme, bits = SCHEMES[i % len(SCHEMES)]
    lens = [int(r.integers(1, 2600)) for _ in range(int(r.integers(1, 9)))]
    wl = W.Workload(f"rsweep{i}", 1, group * hkv, hkv, lens, shuffle_pages=bool(r.random() < 0.5), seed=130 + i)
    layer = int(r.integers(0, 28))
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, hkv, wl.num_pages, scheme, bits, 0, 30 + i)
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
        assert torch.equal(x, y)
    meter_raw = res[2].cpu().numpy()
    tau = float(np.median(meter_raw)) * float(r.uniform(0.2, 0.9))
    contrib, pages, n_rep, d_after = wc.repair_select(res[3], res[4], ctx, tau)
    torch.cuda.synchronize()
    contrib, pages, n_rep, d_after = (t.cpu().numpy() for t in (contrib, pages, n_rep, d_after))
    for b, S in enumerate(wl.ctx_lens):
        ref = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, repair_tau=tau)
        n = (S + 15) // 16
        assert_close(contrib[b, :, :n], ref["contrib"], f"contrib[{b}]", atol=1e-6)
        for hq in range(wl.n_q_heads):
            _check_selection(contrib[b, hq, :n], pages[b, hq, :n_rep[b, hq]], n, d_after[b, hq], tau,
                             ref["contrib"][hq])
