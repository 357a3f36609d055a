"""GPU parity of the value side (§3 output bound, §4.2 "Value side and the
joint event"): the stored value witness (never below the oracle's exact
round-up, at most one fp16 step above), value_term / v_max / out_bound against
the oracle, the bound against the true output error, the joint gate bit for
bit, and the rest of the call identical to the plain one."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, descs, gpu_cache_to_numpy, make_inputs, numpy_cache_to_gpu

pytestmark = pytest.mark.gpu


def _setup(wl, scheme, layer, seed, bits=8):
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, scheme, bits, 0, seed)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    return bt, sm, k, v, q, od, gd, ocache


@pytest.mark.parametrize("scheme", [0, 1])
def test_value_witness_write(scheme):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("w", 1, 28, 4, [1000, 333, 17], shuffle_pages=True, seed=2)
    bt, sm, k, v, q, od, gd, ocache = _setup(wl, scheme, 2, 4)
    gcache = wc.LayerCache.empty(gd, value_witness=True)
    wc.kv_quantize_witness(gd, 2, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache)
    plain = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 2, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), plain)
    torch.cuda.synchronize()
    g, p = gpu_cache_to_numpy(gcache), gpu_cache_to_numpy(plain)
    for name in p:
        assert np.array_equal(g[name].view(np.uint8), p[name].view(np.uint8)), name   # nothing else changes
    gw = g["v_witness"].astype(np.float64)
    ow = ocache["v_witness"].astype(np.float64)
    up = (ocache["v_witness"].view(np.uint16) + 1).view(np.float16).astype(np.float64)
    assert np.all(gw >= ow) and np.all((gw == ow) | (gw == up))


@pytest.mark.parametrize("scheme,bits", [(0, 8), (1, 8), (0, 10)])   # 10-bit: the per-warp plan
def test_value_side_decode_and_joint_gate(scheme, bits):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("d", 1, 28, 4, [4100, 77, 1, 2500, 16, 999], shuffle_pages=True, seed=6)
    layer = 3
    bt, sm, k, v, q, od, gd, ocache = _setup(wl, scheme, layer, 7, bits)
    gcache = numpy_cache_to_gpu(ocache, gd, value_witness=True)     # identical stored inputs on both sides
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    res = wc.metered_decode_attention_v(gd, layer, qd, btd, ctx, gcache, ws)
    plain = wc.metered_decode_attention(gd, layer, qd, btd, ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    for x, y in zip(plain, res[:3]):
        assert torch.equal(x, y)
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    ref = {n: [] for n in ("value_term", "v_max", "out_bound", "out_err", "meter_raw")}
    for b, S in enumerate(wl.ctx_lens):
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache,
                               k.numpy()[offs[b]:offs[b] + S], v.numpy()[offs[b]:offs[b] + S])
        for n in ref:
            ref[n].append(r[n])
    ref = {n: np.stack(x) for n, x in ref.items()}
    vterm, vmax, bound = (t.cpu().numpy() for t in res[3:])
    assert_close(vterm, ref["value_term"], "value_term")
    assert np.array_equal(vmax.astype(np.float64), ref["v_max"])    # a max of the same stored fp16 values
    assert_close(bound, ref["out_bound"], "out_bound")
    assert_sound(vterm, ref["value_term"], None, "value_term")       # rounded up like the meter
    assert np.all(bound >= ref["out_err"])                            # the bound holds on the GPU's numbers
    # the joint gate on the GPU's numbers against the oracle's joint gate on its own
    # fp64 numbers; cells within 1e-3 of either threshold are excluded and counted
    o_raw = ref["meter_raw"].reshape(-1)
    o_vt, o_vm = ref["value_term"].reshape(-1), ref["v_max"].reshape(-1)
    for tk, tv in ((0.1, 0.01), (0.5, 0.05), (1.0, 1e-3), (float(np.median(o_raw)), float(np.median(o_vt / o_vm)))):
        keep_q, keep_kv, kept = wc.gate_joint(res[2].reshape(-1), res[3].reshape(-1), res[4].reshape(-1),
                                              gd.group, tk, tv)
        oq, _, _, _ = OM.joint_gate(o_raw, o_vt, o_vm, tk, tv, gd.group)
        near = (np.abs(o_raw - tk) < 1e-3 * tk + 1e-5) | (np.abs(o_vt - tv * o_vm) < 1e-3 * tv * o_vm + 1e-5)
        assert int(near.sum()) <= max(1, near.size // 20)
        kq = keep_q.cpu().numpy().astype(bool)
        assert np.array_equal(kq[~near], oq[~near])
        kkv = keep_kv.cpu().numpy().astype(bool)
        assert np.array_equal(kkv, kq.reshape(-1, gd.group).all(axis=1))     # any-of-G fallback
        assert kept.cpu().tolist() == [int(kq.sum()), int(kkv.sum())]
