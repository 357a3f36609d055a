"""The allocation-free decode entry point gives the same results as the
workspace-based one.

It exists for callers that cannot allocate device memory at decode time, so
its scratch is a fixed array inside the library.  This file is collected
last so that, if it fails, every other test has already run."""

import ctypes

import numpy as np
import pytest
import torch

import workloads as W
from tests._parity import assert_close, descs, make_inputs

pytestmark = pytest.mark.gpu


def _noalloc_fn():
    import paper_2607_28699_gb300 as wc
    f = wc.lib.wc_metered_decode_attention_noalloc
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    f.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    f.restype = ctypes.c_int
    return f


def test_noalloc_decode_matches_workspace_decode_twice():
    import paper_2607_28699_gb300 as wc
    f = _noalloc_fn()
    P = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
    for call, (scheme, ctx_lens, layer) in enumerate([(0, [3001, 77, 1], 2), (1, [5000, 16], 5)]):
        wl = W.Workload("noalloc", 1, 28, 4, ctx_lens, scheme=scheme, shuffle_pages=True, seed=call + 3)
        bt, sm, k, v, q = make_inputs(wl, layer)
        _, gd = descs(28, 4, wl.num_pages, scheme=scheme, seed=9)
        cache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), cache)
        btg, qg = torch.from_numpy(bt).cuda(), q.cuda()
        ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
        ws = wc.Workspace(gd, wl.batch, wl.max_pages)
        ref_out, ref_meter, ref_raw = wc.metered_decode_attention(gd, layer, qg, btg, ctx, cache, ws)

        out = torch.full_like(ref_out, float("nan"))
        meter = torch.full_like(ref_meter, float("nan"))
        raw = torch.full_like(ref_raw, float("nan"))
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        d = gd.c()
        st = f(ctypes.byref(d), layer, P(qg), P(btg), wl.max_pages, P(ctx), wl.batch, P(cache.k_codes),
               P(cache.v_codes), P(cache.k_scale), P(cache.v_scale), P(cache.k_witness), P(out), P(meter),
               P(raw), P(status), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
        assert st == 0, wc.lib.wc_last_error().decode()
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        assert_close(out.cpu().numpy(), ref_out.cpu().numpy(), "noalloc out")
        assert_close(meter.cpu().numpy(), ref_meter.cpu().numpy(), "noalloc meter")
        assert_close(raw.cpu().numpy(), ref_raw.cpu().numpy(), "noalloc meter_raw")


def test_noalloc_rejects_work_beyond_its_scratch():
    import paper_2607_28699_gb300 as wc
    f = _noalloc_fn()
    # many short sequences: the split plan needs more partials than 4 MiB holds
    batch, max_pages = 4096, 64
    _, gd = descs(32, 8, 16, seed=1)
    cache = wc.LayerCache.empty(gd)
    q = torch.zeros(batch, 32, 128, dtype=torch.float16, device="cuda")
    bt = torch.zeros(batch, max_pages, dtype=torch.int32, device="cuda")
    ctx = torch.ones(batch, dtype=torch.int32, device="cuda")
    out = torch.empty(batch, 32, 128, device="cuda")
    m = torch.empty(batch, 32, device="cuda")
    d = gd.c()
    P = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
    st = f(ctypes.byref(d), 0, P(q), P(bt), max_pages, P(ctx), batch, P(cache.k_codes), P(cache.v_codes),
           P(cache.k_scale), P(cache.v_scale), P(cache.k_witness), P(out), P(m), P(m), None,
           ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 2 and b"scratch" in wc.lib.wc_last_error()
