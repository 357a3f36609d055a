"""The allocation-free decode entry point (wc_metered_decode_attention_noalloc)
gives the same results as the workspace-based one, bit for bit, and matches
the oracle.

It exists for callers that cannot allocate device memory at decode time (a
runtime that pre-plans every buffer, code inside an allocator's own hooks, a
process under a fixed memory budget), so its scratch is a fixed array inside
the library.  This file is collected last so that, if it fails, every other
test has already run."""

import ctypes

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, descs, make_inputs, numpy_cache_to_gpu

pytestmark = pytest.mark.gpu


def _noalloc_fn():
    import paper_2607_28699_gb300 as wc
    f = wc.lib.wc_metered_decode_attention_noalloc
    vp, i32 = ctypes.c_void_p, ctypes.c_int32
    f.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    f.restype = ctypes.c_int
    return f


def _P(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


# batch 1 runs the split plan (partials per (KV head, split) in the scratch),
# several sequences the flattened plan; both schemes
CASES = [(0, [20011], 4), (1, [9000], 1), (0, [3001, 77, 1], 2), (1, [5000, 16], 5)]


@pytest.mark.parametrize("scheme,ctx_lens,layer", CASES)
def test_noalloc_decode_matches_workspace_and_oracle_twice(scheme, ctx_lens, layer):
    import paper_2607_28699_gb300 as wc
    f = _noalloc_fn()
    wl = W.Workload("noalloc", 1, 28, 4, ctx_lens, scheme=scheme, shuffle_pages=True, seed=layer + 3)
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(28, 4, wl.num_pages, scheme=scheme, seed=9)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    cache = numpy_cache_to_gpu(ocache, gd)          # the oracle's stored cache on both sides
    btg, qg = torch.from_numpy(bt).cuda(), q.cuda()
    ctx = torch.tensor(ctx_lens, dtype=torch.int32, device="cuda")
    ws = wc.Workspace(gd, wl.batch, wl.max_pages)
    ref_out, ref_meter, ref_raw = wc.metered_decode_attention(gd, layer, qg, btg, ctx, cache, ws)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    d = gd.c()
    for _ in range(2):                              # two calls in a row share the scratch
        out = torch.full_like(ref_out, float("nan"))
        meter = torch.full_like(ref_meter, float("nan"))
        raw = torch.full_like(ref_raw, float("nan"))
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        st = f(ctypes.byref(d), layer, _P(qg), _P(btg), wl.max_pages, _P(ctx), wl.batch, _P(cache.k_codes),
               _P(cache.v_codes), _P(cache.k_scale), _P(cache.v_scale), _P(cache.k_witness), _P(out),
               _P(meter), _P(raw), _P(status), stream)
        assert st == 0, wc.lib.wc_last_error().decode()
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        for a, b in ((out, ref_out), (meter, ref_meter), (raw, ref_raw)):
            assert torch.equal(a, b)                # same kernels, same plan
    for b, S in enumerate(ctx_lens):
        r = OP.decode_sequence(od, layer, q.numpy()[b], bt[b], S, ocache)
        assert_close(out[b].cpu().numpy(), r["out"], f"noalloc out[{b}]")
        assert_close(raw[b].cpu().numpy(), r["meter_raw"], f"noalloc meter_raw[{b}]")
        assert_sound(raw[b].cpu().numpy(), r["meter_raw"], None, f"noalloc meter_raw[{b}]")


def test_noalloc_rejects_work_beyond_its_scratch_and_a_null_status():
    import paper_2607_28699_gb300 as wc
    f = _noalloc_fn()
    # many short sequences: the plan needs more partials than 16 MiB holds
    batch, max_pages = 4096, 64
    _, gd = descs(32, 8, 16, seed=1)
    cache = wc.LayerCache.empty(gd)
    q = torch.zeros(batch, 32, 128, dtype=torch.float16, device="cuda")
    bt = torch.zeros(batch, max_pages, dtype=torch.int32, device="cuda")
    ctx = torch.ones(batch, dtype=torch.int32, device="cuda")
    out = torch.empty(batch, 32, 128, device="cuda")
    m = torch.empty(batch, 32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = gd.c()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    args = [ctypes.byref(d), 0, _P(q), _P(bt), max_pages, _P(ctx), batch, _P(cache.k_codes), _P(cache.v_codes),
            _P(cache.k_scale), _P(cache.v_scale), _P(cache.k_witness), _P(out), _P(m), _P(m)]
    st = f(*args, _P(status), stream)
    assert st == 2 and b"scratch" in wc.lib.wc_last_error()
    st = f(*args, None, stream)                     # the status word is required
    assert st == 1 and b"dev_status" in wc.lib.wc_last_error()
