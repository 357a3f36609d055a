"""GPU parity of the decode step with the write of its new token fused in
(wc_metered_decode_attention_append): the cache and the outputs are bit for
bit those of wc_kv_quantize_witness followed by wc_metered_decode_attention
(new tokens in the middle of a page, on the first and last slot of a page,
one-token contexts, sequences without a new token, shuffled pages); the
output against the oracle; a slot that is not the context's last is
reported and not written."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, make_inputs

pytestmark = pytest.mark.gpu


def _setup(ctx_lens, seed):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("ap", 1, 28, 4, ctx_lens, shuffle_pages=True, seed=seed)
    bt, sm, k, v, q = make_inputs(wl, 1)
    last = np.cumsum(wl.ctx_lens) - 1                     # each sequence's newest token
    prefix = np.setdiff1d(np.arange(len(sm)), last)
    gd = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=7)
    base = wc.LayerCache.empty(gd)
    kd, vd, smd = k.cuda(), v.cuda(), torch.from_numpy(sm).cuda()
    pi = torch.from_numpy(prefix).cuda()
    wc.kv_quantize_witness(gd, 1, kd[pi].contiguous(), vd[pi].contiguous(), smd[pi].contiguous(), base)
    li = torch.from_numpy(last).cuda()
    return wc, wl, gd, bt, sm, k, v, q, base, kd[li].contiguous(), vd[li].contiguous(), smd[li].contiguous()


def _clone(wc, c):
    return wc.LayerCache(c.k_codes.clone(), c.v_codes.clone(), c.k_scale.clone(), c.v_scale.clone(),
                         c.k_witness.clone())


@pytest.mark.parametrize("ctx_lens,seed", [([4100, 77, 1, 2500, 16, 17, 999], 3), ([32768], 4), ([1, 2, 15, 33], 5)])
def test_append_equals_write_then_decode(ctx_lens, seed):
    wc, wl, gd, bt, sm, k, v, q, base, k_new, v_new, s_new = _setup(ctx_lens, seed)
    if len(ctx_lens) > 3:
        s_new[2] = -1                                      # no new token for one sequence
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    qd, btd = q.cuda(), torch.from_numpy(bt).cuda()
    a, b = _clone(wc, base), _clone(wc, base)
    ws_a, ws_b = wc.Workspace(gd, wl.batch, wl.max_pages), wc.Workspace(gd, wl.batch, wl.max_pages)
    wc.kv_quantize_witness(gd, 1, k_new, v_new, s_new, a)
    ra = wc.metered_decode_attention(gd, 1, qd, btd, ctx, a, ws_a)
    rb = wc.metered_decode_attention_append(gd, 1, qd, btd, ctx, b, ws_b, k_new, v_new, s_new)
    torch.cuda.synchronize()
    assert wc.read_status(ws_a) == 0 and wc.read_status(ws_b) == 0
    for name in ("k_codes", "v_codes", "k_scale", "v_scale", "k_witness"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
    for x, y in zip(ra, rb):
        assert torch.equal(x, y)


def test_append_against_the_oracle():
    wc, wl, gd, bt, sm, k, v, q, base, k_new, v_new, s_new = _setup([700, 33, 16], 6)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    out, meter, raw = wc.metered_decode_attention_append(gd, 1, q.cuda(), torch.from_numpy(bt).cuda(), ctx, base,
                                                         ws, k_new, v_new, s_new)
    torch.cuda.synchronize()
    od = OP.Desc(num_q_heads=28, num_kv_heads=4, num_pages=wl.num_pages, seed=7)
    oc = OP.empty_cache(od)
    OP.write_tokens(od, 1, k.numpy(), v.numpy(), sm, oc)
    for b, S in enumerate(wl.ctx_lens):
        r = OP.decode_sequence(od, 1, q.numpy()[b], bt[b], S, oc)
        assert_close(out[b].cpu().numpy(), r["out"], f"out[{b}]")
        assert_close(raw[b].cpu().numpy(), r["meter_raw"], f"meter_raw[{b}]")


def test_append_slot_not_the_last_is_reported_and_not_written():
    wc, wl, gd, bt, sm, k, v, q, base, k_new, v_new, s_new = _setup([300, 40], 8)
    ctx = torch.tensor(wl.ctx_lens, dtype=torch.int32, device="cuda")
    bad = s_new.clone()
    bad[0] = int(sm[0])                                    # the first token's slot: not the context's last
    c = _clone(wc, base)
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    wc.metered_decode_attention_append(gd, 1, q.cuda(), torch.from_numpy(bt).cuda(), ctx, c, ws, k_new, v_new, bad)
    torch.cuda.synchronize()
    assert wc.read_status(ws) & wc.DEV_BAD_APPEND
    page, off = int(sm[0]) // 16, int(sm[0]) % 16
    assert torch.equal(c.k_codes[page, :, off], base.k_codes[page, :, off])   # untouched
    ref = _clone(wc, base)
    wc.kv_quantize_witness(gd, 1, k_new[1:].contiguous(), v_new[1:].contiguous(), s_new[1:].contiguous(), ref)
    assert torch.equal(c.k_codes, ref.k_codes)            # the other sequence's token is written
