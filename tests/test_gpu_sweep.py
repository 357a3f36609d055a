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
