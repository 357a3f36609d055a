"""Failure detection on the GPU without a fault: a decode whose one page is
never staged makes the warp-specialized kernel's bounded waits run out.

The consumer waiting for the page and then its producer give up after a short
limit, set WC_DEV_TIMEOUT in the workspace's status word and finish (the
copies they had issued land before the kernel exits).  The host reads the
bit; the context stays usable, and the next ordinary call on the same
workspace and cache gives the same results as before, bit for bit."""

import ctypes

import numpy as np
import pytest
import torch

import workloads as W
from tests._parity import descs, make_inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("ctx,stall_page", [(20011, 0), (20011, 700), (3001, 187)])
def test_stalled_page_sets_timeout_and_the_context_stays_usable(ctx, stall_page):
    import paper_2607_28699_gb300 as wc
    wl = W.Workload("stall", 1, 28, 4, [ctx], seed=21)
    bt, sm, k, v, q = make_inputs(wl, 0)
    _, gd = descs(28, 4, wl.num_pages, seed=4)
    cache = wc.LayerCache.empty(gd)
    wc.kv_quantize_witness(gd, 0, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
    btg, qg = torch.from_numpy(bt).cuda(), q.cuda()
    ctxg = torch.tensor([ctx], dtype=torch.int32, device="cuda")
    ws = wc.Workspace(gd, 1, wl.max_pages)
    before = wc.metered_decode_attention(gd, 0, qg, btg, ctxg, cache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0

    out, meter, raw = (torch.empty_like(t) for t in before)
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    d = gd.c()
    st = wc.lib.wc_testing_decode_stalled_page(
        ctypes.byref(d), 0, P(qg), P(btg), wl.max_pages, P(ctxg), P(cache.k_codes), P(cache.v_codes),
        P(cache.k_scale), P(cache.v_scale), P(cache.k_witness), P(out), P(meter), P(raw), ws.ptr(), ws.nbytes,
        stall_page, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, wc.lib.wc_last_error().decode()
    torch.cuda.synchronize()                                   # the kernel returns: nothing hangs
    bits = wc.read_status(ws)
    assert bits & wc.DEV_TIMEOUT, bits
    assert bits & ~(wc.DEV_TIMEOUT) == 0, bits                 # nothing else went wrong

    after = wc.metered_decode_attention(gd, 0, qg, btg, ctxg, cache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    for a, b in zip(before, after):
        assert torch.equal(a, b)


def test_stalled_page_argument_checks():
    import paper_2607_28699_gb300 as wc
    _, gd = descs(28, 4, 4, seed=4)
    d = gd.c()
    f = wc.lib.wc_testing_decode_stalled_page
    args = [ctypes.byref(d), 0, None, None, 4, None, None, None, None, None, None, None, None, None, None, 0]
    assert f(*args, 4, None) == 1                               # stall_page outside [0, max_pages)
    _, g10 = descs(28, 4, 4, bits=10, seed=4)
    d10 = g10.c()
    assert f(ctypes.byref(d10), *args[1:], 0, None) == 2        # 10-bit dither: another kernel
