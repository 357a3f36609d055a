"""GPU parity of metered decode attention (wc_metered_decode_attention)
against the oracle: outputs, meters and raw meters within 1e-3 relative /
1e-5 absolute; the meter bounds the true TV; device status checks."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, descs, make_inputs, numpy_cache_to_gpu, witness_step_up

pytestmark = pytest.mark.gpu


def _oracle_decode(od, layer, q, bt, ctx_lens, ocache, k=None, v=None, seq_offsets=None):
    outs, meters, raws, tvs = [], [], [], []
    for b, S in enumerate(ctx_lens):
        ke = ve = None
        if k is not None:
            o = seq_offsets[b]
            ke, ve = k[o:o + S], v[o:o + S]
        r = OP.decode_sequence(od, layer, q[b], bt[b], S, ocache, ke, ve)
        outs.append(r["out"]); meters.append(r["meter"]); raws.append(r["meter_raw"]); tvs.append(r["tv"])
    return np.stack(outs), np.stack(meters), np.stack(raws), np.stack(tvs)


def _run(wl, scheme=0, bits=8, layout=0, layer=0, seed=1, gpu_writes=True):
    """GPU decode against the oracle.  With gpu_writes the GPU decodes its own
    write of the cache, whose witness may sit one fp16 step above the oracle's
    (the write rounds it up with a margin, never below); the oracle then also
    decodes its cache with every witness one step up, the upper end of what
    the GPU may have stored, and the GPU meters are checked between the two."""
    import paper_2607_28699_gb300 as wc
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, scheme, bits, layout, seed)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    if gpu_writes:
        gcache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache)
    else:
        gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, layer, q.cuda(), torch.from_numpy(bt).cuda(), ctx,
                                                  gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    o = _oracle_decode(od, layer, q.numpy(), bt, wl.ctx_lens, ocache, k.numpy(), v.numpy(), offs)
    o_up = None
    if gpu_writes:
        up = dict(ocache)
        up["k_witness"] = witness_step_up(ocache["k_witness"])
        o_up = _oracle_decode(od, layer, q.numpy(), bt, wl.ctx_lens, up)
    return (out.cpu().numpy(), meter.cpu().numpy(), raw.cpu().numpy()), o, o_up


def _compare(g, o, o_up=None):
    assert_close(g[0], o[0], "out")
    if o_up is None:   # identical stored inputs
        assert_close(g[1], o[1], "meter")
        assert_close(g[2], o[2], "meter_raw")
        assert_sound(g[2], o[2], o[3], "meter_raw")
    else:              # the GPU's own write: between the oracle's meters for the two witness ends
        assert_sound(g[2], o[2], o[3], "meter_raw")
        assert_close(np.maximum(g[2], o_up[2]), o_up[2], "meter_raw (witness one step up)")
        assert_close(np.maximum(g[1], o_up[1]), o_up[1], "meter (witness one step up)")


@pytest.mark.parametrize("scheme,bits,layout", [(0, 8, 0), (0, 10, 0), (0, 8, 1), (1, 8, 0)])
@pytest.mark.parametrize("gpu_writes", [False, True])
def test_decode_matches_oracle_config1_shape(scheme, bits, layout, gpu_writes):
    wl = W.config(1, ctx_scale=0.5)               # S = 2048 + ragged? (2048) -> also test ragged below
    _compare(*_run(wl, scheme, bits, layout, gpu_writes=gpu_writes))


@pytest.mark.parametrize("ctx", [1, 15, 16, 17, 127, 128, 129, 1000, 3001])
def test_decode_ragged_contexts(ctx):
    wl = W.Workload("r", 1, 8, 2, [ctx], seed=4)
    _compare(*_run(wl))


def test_decode_batch_mixed_shuffled_gqa7():
    wl = W.Workload("m", 1, 28, 4, [4100, 77, 1, 2500, 16, 999], shuffle_pages=True, seed=6)
    for scheme in (0, 1):
        _compare(*_run(wl, scheme=scheme, layer=3))


def test_decode_many_splits_long_context():
    wl = W.Workload("long", 1, 28, 4, [20011], seed=8)
    _compare(*_run(wl, bits=10, layer=5))


@pytest.mark.parametrize("scheme,bits", [(0, 8), (1, 8), (0, 10)])
@pytest.mark.parametrize("ctx_lens,hq,hkv", [
    ([0, 1, 16, 17, 40, 0, 33, 5] * 25, 8, 2),      # 200 short sequences: CTAs walk many segments
    ([3000, 1, 0, 16, 2049, 17, 0, 700], 28, 4),     # one long sequence among short and empty ones
    ([0, 5], 8, 2),
    ([(37 * i) % 41 for i in range(600)], 8, 2),    # more sequences than the CTA's threads: several each
])
def test_decode_flattened_plan_batches(ctx_lens, hq, hkv, scheme, bits):
    """A batch of several sequences: the warp-specialized kernel runs the
    flattened split plan (each CTA an equal share of all units' pages, cut at
    unit boundaries), the per-token kernel (fp8, 10-bit dither) the split plan
    or, for the 10-bit dither when that leaves SMs idle, a flattened plan with a
    share per warp: every sequence against the oracle, empty sequences give
    out = 0 and meter 0."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("f", 1, hq, hkv, ctx_lens, shuffle_pages=True, seed=9)
    bt, sm, k, v, q = make_inputs(wl, 0)
    od, gd = descs(hq, hkv, wl.num_pages, scheme, bits, 0, 3)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k.numpy(), v.numpy(), sm, ocache)
    gcache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, meter, raw = out.cpu().numpy(), meter.cpu().numpy(), raw.cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(ctx_lens)[:-1]])
    ocache_up = dict(ocache)
    ocache_up["k_witness"] = witness_step_up(ocache["k_witness"])
    for b, S in enumerate(ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(meter[b] == 0) and np.all(raw[b] == 0)
            continue
        o = offs[b]
        r = OP.decode_sequence(od, 0, q.numpy()[b], bt[b], S, ocache, k.numpy()[o:o + S], v.numpy()[o:o + S])
        r_up = OP.decode_sequence(od, 0, q.numpy()[b], bt[b], S, ocache_up)
        assert_close(out[b], r["out"], f"out[{b}]")
        assert_sound(raw[b], r["meter_raw"], r["tv"], f"meter_raw[{b}]")   # the GPU's write: see _run
        assert_close(np.maximum(raw[b], r_up["meter_raw"]), r_up["meter_raw"], f"meter_raw[{b}]")
        assert_close(np.maximum(meter[b], r_up["meter"]), r_up["meter"], f"meter[{b}]")


@pytest.mark.parametrize("scheme,bits", [(1, 8), (0, 10)])
def test_decode_per_token_kernel_batch(scheme, bits):
    """A batch on the per-token kernel.  The 10-bit dither here takes the
    flattened plan with one share per warp (the split plan would fill 224 of
    304 CTA slots): each warp walks a contiguous run of the batch's pages
    across sequence boundaries and writes one partial per sequence it touched.
    fp8 keeps the split plan (8 splits, merged one warp per output over the
    splits that hold pages).  Empty and short sequences beside long ones, the
    oracle decoding the same stored cache: every sequence against it, empty
    ones give out = 0 and meter 0."""
    import paper_2607_28699_gb300 as wc
    ctx_lens = [0, 3000, 5, 1200, 0, 16, 2049]
    wl = W.Workload("s", 1, 28, 4, ctx_lens, shuffle_pages=True, seed=12)
    bt, sm, k, v, q = make_inputs(wl, 0)
    od, gd = descs(28, 4, wl.num_pages, scheme, bits, 0, 5)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k.numpy(), v.numpy(), sm, ocache)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    out, meter, raw = out.cpu().numpy(), meter.cpu().numpy(), raw.cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(ctx_lens)[:-1]])
    for b, S in enumerate(ctx_lens):
        if S == 0:
            assert np.all(out[b] == 0) and np.all(meter[b] == 0) and np.all(raw[b] == 0)
            continue
        o = offs[b]
        r = OP.decode_sequence(od, 0, q.numpy()[b], bt[b], S, ocache, k.numpy()[o:o + S], v.numpy()[o:o + S])
        assert_close(out[b], r["out"], f"out[{b}]")
        assert_close(raw[b], r["meter_raw"], f"meter_raw[{b}]")
        assert_close(meter[b], r["meter"], f"meter[{b}]")
        assert_sound(raw[b], r["meter_raw"], r["tv"], f"meter_raw[{b}]")


@pytest.mark.parametrize("bits", [8, 10])   # 10: the per-token kernel's per-warp plan
def test_decode_flattened_plan_bad_ctx_sets_status(bits):
    """Out-of-range context lengths in a batch are clamped and reported."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("fb", 1, 8, 2, [64, 30], seed=2)
    bt, sm, k, v, q = make_inputs(wl)
    od, gd = descs(8, 2, wl.num_pages, bits=bits)
    cache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, 2, wl.max_pages)
    btd = torch.from_numpy(bt).cuda()
    ref = wc.metered_decode_attention(gd, 0, q.cuda(), btd, torch.tensor([64, 30], dtype=torch.int32,
                                                                            device="cuda"), cache, ws)
    ref = [t.clone() for t in ref]
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    for bad in ([-5, 30], [64, 10_000]):
        res = wc.metered_decode_attention(gd, 0, q.cuda(), btd, torch.tensor(bad, dtype=torch.int32, device="cuda"),
                                          cache, ws)
        torch.cuda.synchronize()
        assert wc.read_status(ws) & wc.DEV_BAD_CTX
        keep = 1 if bad[0] < 0 else 0       # the sequence whose length is valid is unaffected
        for name, x, y in zip(("out", "meter", "meter_raw"), res, ref):   # (its pages split differently)
            assert_close(x[keep].cpu().numpy(), y[keep].cpu().numpy().astype(np.float64), name)


def test_decode_zero_context_and_repeat_calls():
    """ctx 0 gives out = 0 and meter 0; the workspace is reusable call after call."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("z", 1, 8, 2, [300, 40], seed=2)
    bt, sm, k, v, q = make_inputs(wl)
    od, gd = descs(8, 2, wl.num_pages)
    cache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, 2, wl.max_pages)
    btg = torch.from_numpy(bt).cuda()
    first = None
    for it in range(3):
        ctx = torch.tensor([300, 0] if it == 1 else [300, 40], dtype=torch.int32, device="cuda")
        out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), btg, ctx, cache, ws)
        torch.cuda.synchronize()
        if it == 1:
            assert torch.all(out[1] == 0) and torch.all(meter[1] == 0) and torch.all(raw[1] == 0)
        elif first is None:
            first = (out.clone(), raw.clone())
        else:
            assert torch.equal(out, first[0]) and torch.equal(raw, first[1])   # deterministic
    assert wc.read_status(ws) == 0


@pytest.mark.parametrize("bits,ctx_lens", [(8, [64]), (10, [64]), (10, [64, 40])])   # [64, 40]: per-warp plan
def test_decode_bad_page_and_bad_ctx_set_status(bits, ctx_lens):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("b", 1, 8, 2, ctx_lens, seed=2)
    bt, sm, k, v, q = make_inputs(wl)
    od, gd = descs(8, 2, wl.num_pages, bits=bits)
    cache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    bt_bad = torch.from_numpy(bt).cuda().clone()
    bt_bad[0, 1] = 10_000
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    wc.metered_decode_attention(gd, 0, q.cuda(), bt_bad, ctx, cache, ws)
    assert wc.read_status(ws) & wc.DEV_BAD_PAGE
    if len(ctx_lens) > 1:
        return
    ctx_bad = torch.tensor([65], dtype=torch.int32, device="cuda")    # > max_pages * 16
    wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx_bad, cache, ws)
    assert wc.read_status(ws) & wc.DEV_BAD_CTX


def test_decode_host_validation():
    import paper_2607_28699_gb300 as wc
    _, gd = descs(8, 2, 4)
    cache = wc.LayerCache.empty(gd)
    q = torch.zeros(1, 8, 128, dtype=torch.float16, device="cuda")
    bt = torch.zeros(1, 4, dtype=torch.int32, device="cuda")
    ctx = torch.ones(1, dtype=torch.int32, device="cuda")
    ws = wc.Workspace(gd, 1, 4)
    small = wc.Workspace(gd, 1, 4)
    small.nbytes = 256
    with pytest.raises(wc.WitCertError) as e:
        wc.metered_decode_attention(gd, 0, q, bt, ctx, cache, small)
    assert e.value.status == 4
    bad = wc.CacheDesc(num_q_heads=12, num_kv_heads=8, num_pages=4)
    with pytest.raises(wc.WitCertError):
        wc.metered_decode_attention(bad, 0, q, bt, ctx, cache, ws)
    wide = wc.CacheDesc(num_q_heads=36, num_kv_heads=2, num_pages=4)   # G = 18 > 8
    with pytest.raises(wc.WitCertError) as e:
        wc.metered_decode_attention(wide, 0, q, bt, ctx, cache, ws)
    assert e.value.status == 2


@pytest.mark.parametrize("ctx_lens", [[100, 40], [37]])
def test_decode_zero_value_rows(ctx_lens):
    """Value rows that are exactly zero have scale 0: pages whose every value
    scale is 0 (the first pages of a sequence, or all of it) leave the P scale
    unset until a positive one arrives; outputs and meters match the oracle."""
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("zv", 1, 8, 2, ctx_lens, shuffle_pages=True, seed=12)
    bt, sm, k, v, q = make_inputs(wl, 0)
    v = v.clone()
    v[:20] = 0                                   # the first page and a half of sequence 0
    if len(ctx_lens) > 1:
        v[ctx_lens[0]:] = 0                      # all of sequence 1
    od, gd = descs(8, 2, wl.num_pages, seed=5)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k.numpy(), v.numpy(), sm, ocache)
    gcache = numpy_cache_to_gpu(ocache, gd)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    out, meter, raw = wc.metered_decode_attention(gd, 0, q.cuda(), torch.from_numpy(bt).cuda(), ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    offs = np.concatenate([[0], np.cumsum(ctx_lens)[:-1]])
    for b, S in enumerate(ctx_lens):
        r = OP.decode_sequence(od, 0, q.numpy()[b], bt[b], S, ocache, k.numpy()[offs[b]:offs[b] + S],
                               v.numpy()[offs[b]:offs[b] + S])
        assert np.all(np.isfinite(out[b].cpu().numpy()))
        assert_close(out[b].cpu().numpy(), r["out"], f"out[{b}]")
        assert_close(raw[b].cpu().numpy(), r["meter_raw"], f"meter_raw[{b}]")
        assert_sound(raw[b].cpu().numpy(), r["meter_raw"], r["tv"], f"meter_raw[{b}]")
