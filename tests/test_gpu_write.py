"""GPU parity of the write path (wc_kv_quantize_witness) against the oracle:
bit-exact codes and scales, witness within one fp16 ulp above the exactly
rounded-up norm (never below)."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import pipeline as OP
from tests._parity import assert_close, descs, gpu_cache_to_numpy, make_inputs

pytestmark = pytest.mark.gpu


def _run_both(wl, scheme, bits, layout, layer=0, seed=3):
    import paper_2607_28699_gb300 as wc
    bt, sm, k, v, q = make_inputs(wl, layer)
    od, gd = descs(wl.n_q_heads, wl.n_kv_heads, wl.num_pages, scheme, bits, layout, seed)
    ocache = OP.empty_cache(od)
    OP.write_tokens(od, layer, k.numpy(), v.numpy(), sm, ocache)
    gcache = wc.LayerCache.empty(gd)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    wc.kv_quantize_witness(gd, layer, k.cuda(), v.cuda(), torch.from_numpy(sm).cuda(), gcache,
                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return ocache, gpu_cache_to_numpy(gcache)


def _compare(ocache, gcache):
    for name in ("k_codes", "v_codes", "k_scale", "v_scale"):
        if name in ocache:
            a, b = ocache[name].view(np.uint8), gcache[name].view(np.uint8)
            assert np.array_equal(a, b), f"{name}: {int((a != b).sum())} bytes differ"
    ow = ocache["k_witness"].astype(np.float64)
    gw = gcache["k_witness"].astype(np.float64)
    assert np.all(gw >= ow), "witness below the exact rounded-up norm"
    with np.errstate(invalid="ignore"):   # the step above +inf is a NaN pattern, never equal: inf matches gw == ow
        ulp_up = (ocache["k_witness"].view(np.uint16) + 1).view(np.float16).astype(np.float64)
    assert np.all((gw == ow) | (gw == ulp_up)), "witness more than one ulp above"
    assert_close(gw, ow, "witness")


@pytest.mark.parametrize("scheme,bits,layout", [(0, 8, 0), (0, 10, 0), (0, 8, 1), (1, 8, 0), (1, 8, 1)])
def test_write_matches_oracle_config1_shape(scheme, bits, layout):
    wl = W.config(1, ctx_scale=0.3)               # 1229 tokens: ragged last page
    _compare(*_run_both(wl, scheme, bits, layout))


def test_write_matches_oracle_paged_shuffled_gqa7():
    wl = W.Workload("w", 2, 28, 4, [333, 1000, 17], shuffle_pages=True, seed=5)
    _compare(*_run_both(wl, 0, 8, 0, layer=1))


def test_write_edge_rows():
    """All-zero rows (s = 0), tiny rows (s rounds to 0 -> least subnormal,
    clipping possible), rows at the fp16 range, exact ties, skipped slots."""
    import paper_2607_28699_gb300 as wc
    n = 64
    rng = np.random.default_rng(9)
    k = (rng.normal(size=(n, 2, 128))).astype(np.float16)
    k[0] = 0
    k[1] = np.float16(2.0 ** -24)
    k[2, :, :5] = np.float16(3e-6)
    k[3] = np.float16(60000.0) * np.sign(rng.normal(size=(2, 128))).astype(np.float16)
    k[4] = (rng.normal(size=(2, 128)) * 1e-4).astype(np.float16)
    v = k[::-1].copy()
    slots = np.arange(n, dtype=np.int32) * 3 % 80
    slots[10] = -1
    slots[11] = -7
    for scheme, bits in [(0, 8), (0, 10), (1, 8)]:
        od, gd = descs(4, 2, 5, scheme, bits, 0, seed=77)
        ocache = OP.empty_cache(od)
        OP.write_tokens(od, 2, k, v, slots, ocache)
        gcache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, 2, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                               torch.from_numpy(slots).cuda(), gcache)
        torch.cuda.synchronize()
        _compare(ocache, gpu_cache_to_numpy(gcache))


def test_write_scale_every_fp16_exponent():
    """Rows whose amax takes fp16 values across every exponent (subnormals to
    65504, 64 mantissas each, the largest and smallest included): the scale's
    quotient and the reciprocal behind the fast rounding pass, checked on the
    device through bit-exact scales and codes."""
    import paper_2607_28699_gb300 as wc
    rng = np.random.default_rng(21)
    bits = []
    for e in range(31):
        mant = np.unique(np.concatenate([[0, 1, 1023], rng.integers(0, 1024, size=61)]))[:64]
        bits.extend(int((e << 10) | int(m)) for m in mant)
    amax = np.array(bits, dtype=np.uint16).view(np.float16).astype(np.float64)
    amax = amax[amax > 0]
    n = (amax.size + 1) // 2
    amax = np.resize(amax, 2 * n).reshape(n, 2)
    x = rng.normal(size=(n, 2, 128)) * (amax[..., None] / 3.0)
    x = np.clip(x, -amax[..., None], amax[..., None]).astype(np.float16)
    x = np.clip(x.astype(np.float64), -amax[..., None], amax[..., None])
    idx = rng.integers(0, 128, size=(n, 2))
    sign = np.where(rng.random((n, 2)) < 0.5, -1.0, 1.0)
    np.put_along_axis(x, idx[..., None], (sign * amax)[..., None], axis=2)
    k = x.astype(np.float16)
    assert np.array_equal(np.abs(k.astype(np.float64)).max(axis=2), amax)
    v = k[::-1].copy()
    slots = np.arange(n, dtype=np.int32)
    num_pages = (n + 15) // 16
    for bits_ in (8, 10):
        od, gd = descs(4, 2, num_pages, 0, bits_, 0, seed=29)
        ocache = OP.empty_cache(od)
        OP.write_tokens(od, 1, k, v, slots, ocache)
        gcache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, 1, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                               torch.from_numpy(slots).cuda(), gcache)
        torch.cuda.synchronize()
        _compare(ocache, gpu_cache_to_numpy(gcache))


@pytest.mark.parametrize("n_tok", [1, 5, 15, 16, 17])
@pytest.mark.parametrize("hkv", [1, 4, 8])
def test_write_small_batches_match_oracle(n_tok, hkv):
    """Decode-step sized writes (one index over (token, head) units below 16
    tokens, a per-head grid from 16 on), scattered slots, both schemes."""
    import paper_2607_28699_gb300 as wc
    rng = np.random.default_rng(100 * n_tok + hkv)
    k = (rng.normal(size=(n_tok, hkv, 128)) * rng.lognormal(0, 0.5, size=128)).astype(np.float16)
    v = (rng.normal(size=(n_tok, hkv, 128)) * rng.lognormal(0, 0.5, size=128)).astype(np.float16)
    slots = rng.permutation(6 * 16)[:n_tok].astype(np.int32)
    for scheme, bits in [(0, 8), (1, 8)]:
        od, gd = descs(hkv, hkv, 6, scheme, bits, 0, seed=11)
        ocache = OP.empty_cache(od)
        OP.write_tokens(od, 3, k, v, slots, ocache)
        gcache = wc.LayerCache.empty(gd)
        wc.kv_quantize_witness(gd, 3, torch.from_numpy(k).cuda(), torch.from_numpy(v).cuda(),
                               torch.from_numpy(slots).cuda(), gcache)
        torch.cuda.synchronize()
        _compare(ocache, gpu_cache_to_numpy(gcache))


def test_write_bad_slot_sets_status_and_skips():
    import paper_2607_28699_gb300 as wc
    od, gd = descs(4, 2, 2, 0, 8, 0)
    k = torch.randn(3, 2, 128, dtype=torch.float16, device="cuda")
    slots = torch.tensor([0, 32, 5], dtype=torch.int32, device="cuda")   # 32 = past the pool
    cache = wc.LayerCache.empty(gd)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    wc.kv_quantize_witness(gd, 0, k, k, slots, cache, dev_status=status)
    assert wc.read_status(status) == wc.DEV_BAD_SLOT
    assert int(cache.k_codes[0, :, 5].abs().sum()) > 0


def test_write_host_validation():
    import paper_2607_28699_gb300 as wc
    _, gd = descs(4, 2, 2, 0, 8, 0)
    cache = wc.LayerCache.empty(gd)
    k = torch.zeros(1, 2, 128, dtype=torch.float16, device="cuda")
    s = torch.zeros(1, dtype=torch.int32, device="cuda")
    bad = wc.CacheDesc(num_q_heads=4, num_kv_heads=2, num_pages=2, dither_bits=9)
    with pytest.raises(wc.WitCertError):
        wc.kv_quantize_witness(bad, 0, k, k, s, cache)
    with pytest.raises(wc.WitCertError):
        wc.kv_quantize_witness(gd, 70000, k, k, s, cache)
    fp8 = wc.CacheDesc(num_q_heads=4, num_kv_heads=2, num_pages=2, scheme=wc.SCHEME_FP8_E4M3)
    with pytest.raises(wc.WitCertError):      # scales must be NULL for fp8
        wc.kv_quantize_witness(fp8, 0, k, k, s, cache)
