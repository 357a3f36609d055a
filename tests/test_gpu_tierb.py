"""GPU parity of the Tier-B certificate (wc_metered_decode_attention_tier_b,
§4.2) against the oracle: meter_b / meter_b_raw within 1e-3 relative / 1e-5
absolute, and the rest of the call identical to wc_metered_decode_attention."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, descs, make_inputs

pytestmark = pytest.mark.gpu


def _run(wl, bits=8, layout=0, layer=0, seed=1, delta=1e-6):
    import paper_2607_28699_gb300 as wc
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, 0, bits, layout, seed)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    gcache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    res_b = wc.metered_decode_attention_tier_b(gd, layer, qd, btd, ctx, gcache, ws, delta)
    res_a = wc.metered_decode_attention(gd, layer, qd, btd, ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    for x, y in zip(res_a, res_b[:3]):              # same output and Tier-A meters, bit for bit
        assert torch.equal(x, y)
    mb, mbr = [], []
    for b, S in enumerate(wl.ctx_lens):
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache, delta_loc=delta)
        mb.append(r["meter_b"]); mbr.append(r["meter_b_raw"])
    assert_close(res_b[4].cpu().numpy(), np.stack(mbr), "meter_b_raw")
    assert_sound(res_b[4].cpu().numpy(), np.stack(mbr), None, "meter_b_raw")
    assert_close(res_b[3].cpu().numpy(), np.stack(mb), "meter_b")


@pytest.mark.parametrize("bits,layout", [(8, 0), (10, 0), (8, 1)])
def test_tier_b_matches_oracle_config1_shape(bits, layout):
    _run(W.config(1, ctx_scale=0.3), bits, layout)


@pytest.mark.parametrize("bits", [8, 10])   # the 10-bit dither: the per-token kernel's per-warp plan
@pytest.mark.parametrize("delta", [1e-2, 1e-9])
def test_tier_b_batch_mixed_shuffled_gqa7(delta, bits):
    wl = W.Workload("m", 1, 28, 4, [4100, 77, 1, 2500, 16, 999], shuffle_pages=True, seed=6)
    _run(wl, bits=bits, layer=3, delta=delta)


def test_tier_b_many_splits():
    wl = W.Workload("l", 1, 8, 2, [40000], seed=8)
    _run(wl, layer=1)
