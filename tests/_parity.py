"""Shared helpers for the GPU parity tests: run the oracle and the CUDA path
on the same seeded inputs and compare."""

import numpy as np
import torch

import workloads as W
from oracle import pipeline as OP

RTOL, ATOL = 1e-3, 1e-5     # fp32 outputs, meters, band norms


def close(gpu, ref, rtol=RTOL, atol=ATOL):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    both_inf = np.isinf(gpu) & np.isinf(ref) & (np.sign(gpu) == np.sign(ref))
    with np.errstate(invalid="ignore"):   # inf - inf: judged by both_inf
        ok = both_inf | (np.abs(gpu - ref) <= atol + rtol * np.abs(ref))
    return ok


def margin(gpu, ref, rtol=RTOL, atol=ATOL):
    """Largest |gpu - ref| / (atol + rtol |ref|) over finite entries (1.0 = at tolerance)."""
    g, r = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    fin = np.isfinite(g) & np.isfinite(r)
    if not np.any(fin):
        return 0.0
    return float(np.max(np.abs(g[fin] - r[fin]) / (atol + rtol * np.abs(r[fin]))))


def assert_close(gpu, ref, what, rtol=RTOL, atol=ATOL):
    print(f"[margin] {what}: {margin(gpu, ref, rtol, atol):.3f}")
    ok = close(gpu, ref, rtol, atol)
    if not np.all(ok):
        g, r = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
        idx = np.argwhere(~ok)[:5]
        raise AssertionError(f"{what}: {int((~ok).sum())}/{ok.size} outside tol; first {idx.tolist()} "
                             f"gpu={g[tuple(idx.T)]} ref={r[tuple(idx.T)]}")


def assert_sound(gpu, ref, tv, what):
    """One-sided soundness of a GPU meter (§3 Thm. "Sound replacement"): on or
    above the oracle's fp64 meter and the true TV, per cell, with no slack."""
    g = np.asarray(gpu, np.float64)
    below = g < np.asarray(ref, np.float64)
    assert not np.any(below), f"{what}: {int(below.sum())} cells below the oracle's fp64 meter"
    if tv is not None:
        under = g < np.asarray(tv, np.float64)
        assert not np.any(under), f"{what}: {int(under.sum())} cells below the true TV"


def witness_step_up(w):
    """Every stored fp16 witness one fp16 step up (0 to the least subnormal):
    the largest value the GPU write may store for it."""
    w = np.asarray(w, dtype=np.float16)
    return (w.view(np.uint16) + 1).view(np.float16)


def descs(n_q, n_kv, num_pages, scheme=0, bits=8, layout=0, seed=0, num_bypass_pairs=0):
    import paper_2607_28699_gb300 as wc
    o = OP.Desc(num_q_heads=n_q, num_kv_heads=n_kv, num_pages=num_pages, scheme=scheme,
                dither_bits=bits, rope_layout=layout, seed=seed, num_bypass_pairs=num_bypass_pairs)
    g = wc.CacheDesc(num_q_heads=n_q, num_kv_heads=n_kv, num_pages=num_pages, scheme=scheme,
                     dither_bits=bits, rope_layout=layout, seed=seed)
    return o, g


def gpu_cache_to_numpy(cache):
    out = {"k_codes": cache.k_codes.cpu().numpy(), "v_codes": cache.v_codes.cpu().numpy(),
           "k_witness": cache.k_witness.cpu().numpy()}
    if cache.k_scale is not None:
        out["k_scale"] = cache.k_scale.cpu().numpy()
        out["v_scale"] = cache.v_scale.cpu().numpy()
    if cache.v_witness is not None:
        out["v_witness"] = cache.v_witness.cpu().numpy()
    if cache.k_bypass is not None:
        out["k_bypass"] = cache.k_bypass.cpu().numpy()
    if cache.bypass_pairs is not None:
        out["bypass_pairs"] = cache.bypass_pairs.cpu().numpy().astype(np.int64)
    return out


def numpy_cache_to_gpu(cache, desc_g, value_witness=False):
    import paper_2607_28699_gb300 as wc
    m = cache["bypass_pairs"].shape[1] if "bypass_pairs" in cache else 0
    c = wc.LayerCache.empty(desc_g, value_witness=value_witness, num_bypass_pairs=m)
    if m:
        c.k_bypass.copy_(torch.from_numpy(cache["k_bypass"]))
        c.bypass_pairs.copy_(torch.from_numpy(cache["bypass_pairs"].astype(np.int32)))
    if value_witness:
        c.v_witness.copy_(torch.from_numpy(cache["v_witness"]))
    c.k_codes.copy_(torch.from_numpy(cache["k_codes"]))
    c.v_codes.copy_(torch.from_numpy(cache["v_codes"]))
    c.k_witness.copy_(torch.from_numpy(cache["k_witness"]))
    if "k_scale" in cache:
        c.k_scale.copy_(torch.from_numpy(cache["k_scale"]))
        c.v_scale.copy_(torch.from_numpy(cache["v_scale"]))
    return c


def make_inputs(wl, layer=0):
    """CPU-drawn inputs (identical for both sides)."""
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, layer)
    q = W.layer_queries(wl, layer)
    return bt, sm, k, v, q
