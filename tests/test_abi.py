"""The C-ABI library loads and exports every entry point include/witcert.h
declares; host-side argument checks fail before any launch (no GPU needed)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "witcert.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(wc_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    import paper_2607_28699_gb300 as wc
    return wc.lib


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("wc_kv_quantize_witness", "wc_metered_decode_attention", "wc_gate", "wc_workspace_size"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    import paper_2607_28699_gb300 as wc
    assert set(wc.EXPORTS) <= set(_declared())
    assert wc.version() == (1, 0)


def test_host_validation_without_gpu(lib):
    import paper_2607_28699_gb300 as wc
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, dither_bits=9).c()
    st = lib.wc_kv_quantize_witness(ctypes.byref(d), 0, None, None, None, 0, None, None, None, None,
                                    None, None, None)
    assert st == 2 and b"dither_bits" in lib.wc_last_error()
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=3, num_pages=4).c()
    assert lib.wc_kv_quantize_witness(ctypes.byref(d), 0, None, None, None, 0, None, None, None, None,
                                      None, None, None) == 1
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    d.head_dim = 64
    assert lib.wc_metered_decode_attention(ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None,
                                           None, None, None, None, None, None, 0, None) == 2
    assert lib.wc_gate(None, 7, 2, ctypes.c_float(0.1), None, None, None, None) == 1
    assert lib.wc_kv_quantize_witness(None, 0, None, None, None, 0, None, None, None, None,
                                      None, None, None) == 1


def test_tier_b_host_validation_without_gpu(lib):
    """Tier B is refused before any launch for the fp8 scheme, for delta_loc
    outside (0, 1) and without its output pointers."""
    import paper_2607_28699_gb300 as wc
    f = lib.wc_metered_decode_attention_tier_b
    fp8 = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, scheme=wc.SCHEME_FP8_E4M3).c()
    dummy = ctypes.c_void_p(16)
    args = lambda d, delta, mb: (ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None, None, None,
                                 ctypes.c_double(delta), None, None, None, mb, mb, None, 0, None)
    assert f(*args(fp8, 0.01, dummy)) == 2 and b"Tier B" in lib.wc_last_error()
    int8 = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    for bad in (0.0, 1.0, -0.5, float("nan")):
        assert f(*args(int8, bad, dummy)) == 1 and b"delta_loc" in lib.wc_last_error()
    assert f(*args(int8, 0.01, None)) == 1 and b"meter_b" in lib.wc_last_error()


def test_value_side_host_validation_without_gpu(lib):
    import paper_2607_28699_gb300 as wc
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    assert lib.wc_kv_quantize_witness_v(ctypes.byref(d), 0, None, None, None, 0, None, None, None, None, None,
                                        None, None, None) == 1 and b"v_witness" in lib.wc_last_error()
    assert lib.wc_metered_decode_attention_v(ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None, None,
                                             None, None, None, None, None, None, None, None, None, 0,
                                             None) == 1 and b"v_witness" in lib.wc_last_error()
    assert lib.wc_gate_joint(None, None, None, 4, 2, ctypes.c_float(0.1), ctypes.c_float(0.1), None, None, None,
                             None) == 1


def test_repair_host_validation_without_gpu(lib):
    import paper_2607_28699_gb300 as wc
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    vp = ctypes.c_void_p
    args = lambda pt, sn: (ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None, None, None,
                           None, None, None, pt, sn, None, 0, None)
    assert lib.wc_metered_decode_attention_repair(*args(None, vp(16))) == 1
    assert b"page_terms" in lib.wc_last_error()
    assert lib.wc_metered_decode_attention_repair(*args(vp(4), vp(16))) == 1
    assert b"8-byte aligned" in lib.wc_last_error()
    f = ctypes.c_float(0.1)
    sel = lambda batch, hq, mp, pt=vp(16), sn=vp(16), rp=vp(16): lib.wc_repair_select(
        pt, sn, vp(16), batch, hq, mp, None, f, None, rp, vp(16), vp(16), None, None)
    assert sel(1, 8, 16385) == 2 and b"16384" in lib.wc_last_error()
    assert sel(1, 8, 0) == 1
    assert sel(1, 0, 4) == 1
    assert sel(-1, 8, 4) == 1
    assert sel(0, 8, 4) == 0                      # nothing to select, nothing launched
    assert sel(1, 8, 4, rp=None) == 1 and b"repair_pages" in lib.wc_last_error()
    assert sel(1, 8, 4, sn=vp(12)) == 1 and b"aligned" in lib.wc_last_error()


def test_grouped_scheme_host_validation_without_gpu(lib):
    import paper_2607_28699_gb300 as wc
    vp = ctypes.c_void_p
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, scheme=wc.SCHEME_DITHER_INT8_G32).c()
    # the per-token entry points do not read a grouped cache
    assert lib.wc_kv_quantize_witness(ctypes.byref(d), 0, vp(16), vp(16), vp(16), 1, vp(16), vp(16), vp(16),
                                      vp(16), vp(16), None, None) == 2 and b"_g32" in lib.wc_last_error()
    assert lib.wc_metered_decode_attention(ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None,
                                           None, None, None, None, None, None, 0, None) == 2
    assert lib.wc_metered_decode_attention_noalloc(ctypes.byref(d), 0, None, None, 1, None, 1, None, None, None,
                                                   None, None, None, None, None, None, None) == 2
    g32 = lambda desc, m, kb=vp(16), pr=vp(16): lib.wc_kv_quantize_witness_g32(
        ctypes.byref(desc), 0, vp(16), vp(16), vp(16), 0, vp(16), vp(16), vp(16), vp(16), vp(16), kb, pr, m,
        None, None)
    assert g32(d, 4) == 0                               # no tokens: nothing launched
    assert g32(d, 17) == 1 and b"num_bypass_pairs" in lib.wc_last_error()
    assert g32(d, 4, kb=None) == 1
    assert g32(d, 4, kb=vp(8)) == 1 and b"aligned" in lib.wc_last_error()
    assert g32(d, 0, kb=None, pr=None) == 0
    d0 = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    assert g32(d0, 0) == 1 and b"WC_SCHEME_DITHER_INT8_G32" in lib.wc_last_error()
    d10 = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, scheme=2, dither_bits=10).c()
    assert g32(d10, 0) == 2
    lib.wc_workspace_size(ctypes.byref(d), 1, 8)      # accepted (without a GPU: no device to size for)
    assert b"scheme" not in lib.wc_last_error() and b"_g32" not in lib.wc_last_error()
    sel = lambda n, hkv, layout, m, pairs=vp(16): lib.wc_select_bypass_pairs(vp(16), n, hkv, layout, m, pairs, None)
    assert sel(4, 2, 0, 0) == 0
    assert sel(4, 2, 0, 17) == 1 and sel(4, 0, 0, 4) == 1 and sel(4, 2, 5, 4) == 2 and sel(4, 2, 0, 4, None) == 1


def test_append_host_validation_without_gpu(lib):
    import paper_2607_28699_gb300 as wc
    vp = ctypes.c_void_p
    call = lambda desc, kn=vp(16), vn=vp(16), sn=vp(16): lib.wc_metered_decode_attention_append(
        ctypes.byref(desc), 0, vp(16), vp(16), 1, vp(16), 1, vp(16), vp(16), vp(16), vp(16), vp(16), kn, vn, sn,
        vp(16), vp(16), vp(16), vp(256), 1 << 20, None)
    d = wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4).c()
    assert call(d, sn=None) == 1 and b"slot_new" in lib.wc_last_error()
    assert call(d, kn=vp(8)) == 1 and b"aligned" in lib.wc_last_error()
    for other in (wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, scheme=wc.SCHEME_FP8_E4M3),
                  wc.CacheDesc(num_q_heads=8, num_kv_heads=2, num_pages=4, dither_bits=10)):
        o = other.c()
        assert call(o) == 2 and b"append" in lib.wc_last_error()
