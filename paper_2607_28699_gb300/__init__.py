"""Python binding of the WitCert GB300 library (ctypes over ``include/witcert.h``).

Argument marshalling only: every function passes device pointers, sizes and
the current CUDA stream to the C ABI, where all work runs in the library's
CUDA kernels.  PyTorch supplies device memory and streams.  There is no CPU
fallback: importing this package without the compiled library raises.

    import paper_2607_28699_gb300 as wc
    desc = wc.CacheDesc(num_q_heads=28, num_kv_heads=4, num_pages=n)
    cache = wc.LayerCache.empty(desc, device="cuda")
    wc.kv_quantize_witness(desc, layer, k, v, slot_mapping, cache)
    ws = wc.Workspace(desc, batch, max_pages)
    out, meter, meter_raw = wc.metered_decode_attention(desc, layer, q, block_table,
                                                        ctx_lens, cache, ws)
    keep_q, keep_kv, n_kept = wc.gate(meter_raw, group, tau)
"""

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libwitcert.so")

SCHEME_DITHER_INT8 = 0
SCHEME_FP8_E4M3 = 1
SCHEME_DITHER_INT8_G32 = 2
ROPE_HALF = 0
ROPE_INTERLEAVED = 1
DEV_BAD_SLOT, DEV_BAD_PAGE, DEV_BAD_CTX, DEV_TIMEOUT, DEV_BAD_PAIR, DEV_BAD_APPEND = 1, 2, 4, 8, 16, 32
EXPORTS = ("wc_kv_quantize_witness", "wc_workspace_size", "wc_metered_decode_attention",
           "wc_metered_decode_attention_tier_b", "wc_metered_decode_attention_noalloc",
           "wc_kv_quantize_witness_v", "wc_metered_decode_attention_v", "wc_gate_joint",
           "wc_metered_decode_attention_repair", "wc_repair_select",
           "wc_kv_quantize_witness_g32", "wc_metered_decode_attention_g32", "wc_select_bypass_pairs",
           "wc_metered_decode_attention_append", "wc_testing_decode_stalled_page",
           "wc_gate", "wc_read_status", "wc_last_error", "wc_version")


class WitCertError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"witcert status {status}: {message}")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64
    lib.wc_kv_quantize_witness.argtypes = [vp, i32, vp, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp]
    lib.wc_kv_quantize_witness.restype = ctypes.c_int
    lib.wc_workspace_size.argtypes = [vp, i32, i32]
    lib.wc_workspace_size.restype = ctypes.c_size_t
    lib.wc_metered_decode_attention.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp,
                                                vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.wc_metered_decode_attention.restype = ctypes.c_int
    lib.wc_metered_decode_attention_tier_b.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp,
                                                       ctypes.c_double, vp, vp, vp, vp, vp, vp, ctypes.c_size_t,
                                                       vp]
    lib.wc_metered_decode_attention_tier_b.restype = ctypes.c_int
    lib.wc_testing_decode_stalled_page.argtypes = [vp, i32, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                                   vp, ctypes.c_size_t, i32, vp]
    lib.wc_testing_decode_stalled_page.restype = ctypes.c_int
    lib.wc_gate.argtypes = [vp, i32, i32, ctypes.c_float, vp, vp, vp, vp]
    lib.wc_gate.restype = ctypes.c_int
    lib.wc_gate_joint.argtypes = [vp, vp, vp, i32, i32, ctypes.c_float, ctypes.c_float, vp, vp, vp, vp]
    lib.wc_gate_joint.restype = ctypes.c_int
    lib.wc_kv_quantize_witness_v.argtypes = [vp, i32, vp, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.wc_kv_quantize_witness_v.restype = ctypes.c_int
    lib.wc_metered_decode_attention_v.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp,
                                                  vp, vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.wc_metered_decode_attention_v.restype = ctypes.c_int
    lib.wc_metered_decode_attention_repair.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp,
                                                       vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.wc_metered_decode_attention_repair.restype = ctypes.c_int
    lib.wc_repair_select.argtypes = [vp, vp, vp, i32, i32, i32, vp, ctypes.c_float, vp, vp, vp, vp, vp, vp]
    lib.wc_repair_select.restype = ctypes.c_int
    lib.wc_kv_quantize_witness_g32.argtypes = [vp, i32, vp, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, i32, vp, vp]
    lib.wc_kv_quantize_witness_g32.restype = ctypes.c_int
    lib.wc_metered_decode_attention_g32.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp, vp, i32,
                                                    ctypes.c_double, vp, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.wc_metered_decode_attention_g32.restype = ctypes.c_int
    lib.wc_select_bypass_pairs.argtypes = [vp, i32, i32, i32, i32, vp, vp]
    lib.wc_select_bypass_pairs.restype = ctypes.c_int
    lib.wc_metered_decode_attention_append.argtypes = [vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, vp, vp, vp, vp,
                                                       vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.wc_metered_decode_attention_append.restype = ctypes.c_int
    lib.wc_read_status.argtypes = [vp, i32, vp, vp]
    lib.wc_read_status.restype = ctypes.c_int
    lib.wc_last_error.argtypes = []
    lib.wc_last_error.restype = ctypes.c_char_p
    lib.wc_version.restype = ctypes.c_int32
    del u64
    return lib


lib = _load()


class _Desc(ctypes.Structure):
    _fields_ = [("head_dim", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("num_bands", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("num_pages", ctypes.c_int32),
                ("scheme", ctypes.c_int32), ("rope_layout", ctypes.c_int32),
                ("dither_bits", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("seed", ctypes.c_uint64)]


@dataclass
class CacheDesc:
    """Mirror of ``wc_cache_desc``."""
    num_q_heads: int
    num_kv_heads: int
    num_pages: int
    scheme: int = SCHEME_DITHER_INT8
    rope_layout: int = ROPE_HALF
    dither_bits: int = 8
    seed: int = 0
    head_dim: int = 128
    num_bands: int = 8
    page_size: int = 16

    @property
    def group(self):
        return self.num_q_heads // self.num_kv_heads

    def c(self):
        return _Desc(self.head_dim, self.num_q_heads, self.num_kv_heads, self.num_bands,
                     self.page_size, self.num_pages, self.scheme, self.rope_layout,
                     self.dither_bits, 0, self.seed & (2 ** 64 - 1))


def _check(status):
    if status != 0:
        raise WitCertError(status, lib.wc_last_error().decode())


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to the library must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


@dataclass
class LayerCache:
    """One layer's paged cache tensors (layout in ``include/witcert.h``)."""
    k_codes: torch.Tensor
    v_codes: torch.Tensor
    k_scale: Optional[torch.Tensor]
    v_scale: Optional[torch.Tensor]
    k_witness: torch.Tensor
    v_witness: Optional[torch.Tensor] = None   # (||v^ - v||, ||v||) per slot, value side only
    k_bypass: Optional[torch.Tensor] = None    # grouped scheme: exact bypassed key values [.., 16, 2m]
    bypass_pairs: Optional[torch.Tensor] = None   # grouped scheme: int32 [Hkv, m] RoPE pair set

    @staticmethod
    def empty(desc: CacheDesc, device="cuda", value_witness=False, num_bypass_pairs=0):
        shp = (desc.num_pages, desc.num_kv_heads, desc.page_size)
        code_t = torch.uint8 if desc.scheme == SCHEME_FP8_E4M3 else torch.int8
        grouped = desc.scheme == SCHEME_DITHER_INT8_G32
        sshp = shp + (desc.head_dim // 32,) if grouped else shp
        dither = desc.scheme != SCHEME_FP8_E4M3
        m = num_bypass_pairs if grouped else 0
        return LayerCache(
            torch.zeros(shp + (desc.head_dim,), dtype=code_t, device=device),
            torch.zeros(shp + (desc.head_dim,), dtype=code_t, device=device),
            torch.zeros(sshp, dtype=torch.float16, device=device) if dither else None,
            torch.zeros(sshp, dtype=torch.float16, device=device) if dither else None,
            torch.zeros(shp + (desc.num_bands,), dtype=torch.float16, device=device),
            torch.zeros(shp + (2,), dtype=torch.float16, device=device) if value_witness else None,
            torch.zeros(shp + (2 * m,), dtype=torch.float16, device=device) if m else None,
            torch.zeros(desc.num_kv_heads, m, dtype=torch.int32, device=device) if grouped else None)

    @property
    def num_bypass_pairs(self):
        return 0 if self.bypass_pairs is None else int(self.bypass_pairs.shape[1])

    def nbytes(self):
        return sum(t.numel() * t.element_size() for t in
                   (self.k_codes, self.v_codes, self.k_scale, self.v_scale, self.k_witness, self.v_witness,
                    self.k_bypass)
                   if t is not None)


def kv_quantize_witness(desc: CacheDesc, layer: int, k: torch.Tensor, v: torch.Tensor,
                        slot_mapping: torch.Tensor, cache: LayerCache,
                        dev_status: Optional[torch.Tensor] = None, stream=None):
    """``wc_kv_quantize_witness`` (``_v`` when the cache holds a value witness):
    k, v fp16 [n_tok, Hkv, 128]; slots int32 [n_tok]."""
    d = desc.c()
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        _check(lib.wc_kv_quantize_witness_g32(
            ctypes.byref(d), layer, _ptr(k), _ptr(v), _ptr(slot_mapping), int(slot_mapping.numel()),
            _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
            _ptr(cache.k_witness), _ptr(cache.k_bypass), _ptr(cache.bypass_pairs), cache.num_bypass_pairs,
            _ptr(dev_status), _stream(stream)))
    elif cache.v_witness is None:
        _check(lib.wc_kv_quantize_witness(
            ctypes.byref(d), layer, _ptr(k), _ptr(v), _ptr(slot_mapping), int(slot_mapping.numel()),
            _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
            _ptr(cache.k_witness), _ptr(dev_status), _stream(stream)))
    else:
        _check(lib.wc_kv_quantize_witness_v(
            ctypes.byref(d), layer, _ptr(k), _ptr(v), _ptr(slot_mapping), int(slot_mapping.numel()),
            _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
            _ptr(cache.k_witness), _ptr(cache.v_witness), _ptr(dev_status), _stream(stream)))


def workspace_size(desc: CacheDesc, batch: int, max_pages: int) -> int:
    d = desc.c()
    n = lib.wc_workspace_size(ctypes.byref(d), batch, max_pages)
    if n == 0:
        raise WitCertError(1, lib.wc_last_error().decode())
    return n


class Workspace:
    """Zero-filled device workspace for ``metered_decode_attention``."""

    def __init__(self, desc: CacheDesc, batch: int, max_pages: int, device="cuda"):
        self.nbytes = workspace_size(desc, batch, max_pages)
        self.buf = torch.zeros(self.nbytes + 256, dtype=torch.uint8, device=device)
        off = (-self.buf.data_ptr()) % 256
        self.view = self.buf[off:off + self.nbytes]

    def ptr(self):
        return ctypes.c_void_p(self.view.data_ptr())


def metered_decode_attention(desc: CacheDesc, layer: int, q: torch.Tensor, block_table: torch.Tensor,
                             ctx_lens: torch.Tensor, cache: LayerCache, ws: Workspace,
                             out=None, meter=None, meter_raw=None, stream=None):
    """``wc_metered_decode_attention``; returns (out [B,Hq,128], meter [B,Hq], meter_raw [B,Hq]) fp32."""
    batch, max_pages = block_table.shape
    dev = q.device
    if out is None:
        out = torch.empty(batch, desc.num_q_heads, desc.head_dim, dtype=torch.float32, device=dev)
    if meter is None:
        meter = torch.empty(batch, desc.num_q_heads, dtype=torch.float32, device=dev)
    if meter_raw is None:
        meter_raw = torch.empty(batch, desc.num_q_heads, dtype=torch.float32, device=dev)
    d = desc.c()
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        _decode_g32(d, layer, q, block_table, ctx_lens, cache, ws, 0.0, out, meter, meter_raw, None, None, stream)
        return out, meter, meter_raw
    _check(lib.wc_metered_decode_attention(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), _ptr(out), _ptr(meter), _ptr(meter_raw), ws.ptr(), ws.nbytes,
        _stream(stream)))
    return out, meter, meter_raw


def metered_decode_attention_append(desc: CacheDesc, layer: int, q: torch.Tensor, block_table: torch.Tensor,
                                    ctx_lens: torch.Tensor, cache: LayerCache, ws: Workspace, k_new: torch.Tensor,
                                    v_new: torch.Tensor, slot_new: torch.Tensor, out=None, meter=None,
                                    meter_raw=None, stream=None):
    """``wc_metered_decode_attention_append``: writes each sequence's new token (k_new, v_new fp16
    [B, Hkv, 128] at slot_new int32 [B], the last of its context) and decodes, in one step;
    returns (out, meter, meter_raw)."""
    batch, max_pages = block_table.shape
    dev = q.device
    cells = (batch, desc.num_q_heads)
    out = torch.empty(batch, desc.num_q_heads, desc.head_dim, dtype=torch.float32, device=dev) if out is None else out
    meter = torch.empty(cells, dtype=torch.float32, device=dev) if meter is None else meter
    meter_raw = torch.empty(cells, dtype=torch.float32, device=dev) if meter_raw is None else meter_raw
    d = desc.c()
    _check(lib.wc_metered_decode_attention_append(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), _ptr(k_new), _ptr(v_new), _ptr(slot_new), _ptr(out), _ptr(meter), _ptr(meter_raw),
        ws.ptr(), ws.nbytes, _stream(stream)))
    return out, meter, meter_raw


def _decode_g32(d, layer, q, block_table, ctx_lens, cache, ws, delta_loc, out, meter, meter_raw, meter_b,
                meter_b_raw, stream):
    """``wc_metered_decode_attention_g32`` (grouped-scale cache with the outlier bypass)."""
    batch, max_pages = block_table.shape
    _check(lib.wc_metered_decode_attention_g32(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), _ptr(cache.k_bypass), _ptr(cache.bypass_pairs), cache.num_bypass_pairs,
        float(delta_loc), _ptr(out), _ptr(meter), _ptr(meter_raw), _ptr(meter_b), _ptr(meter_b_raw),
        ws.ptr(), ws.nbytes, _stream(stream)))


def select_bypass_pairs(k: torch.Tensor, m: int, rope_layout: int = ROPE_HALF, pairs=None, stream=None):
    """``wc_select_bypass_pairs``: k fp16 [n_tok, Hkv, 128] -> int32 [Hkv, m], the m RoPE pairs of
    largest energy per KV head in increasing order."""
    n_tok, hkv = k.shape[0], k.shape[1]
    pairs = torch.empty(hkv, m, dtype=torch.int32, device=k.device) if pairs is None else pairs
    _check(lib.wc_select_bypass_pairs(_ptr(k), n_tok, hkv, rope_layout, m, _ptr(pairs), _stream(stream)))
    return pairs


def metered_decode_attention_tier_b(desc: CacheDesc, layer: int, q: torch.Tensor, block_table: torch.Tensor,
                                    ctx_lens: torch.Tensor, cache: LayerCache, ws: Workspace, delta_loc: float,
                                    out=None, meter=None, meter_raw=None, meter_b=None, meter_b_raw=None,
                                    stream=None):
    """``wc_metered_decode_attention_tier_b``; returns (out, meter, meter_raw, meter_b, meter_b_raw)."""
    batch, max_pages = block_table.shape
    dev = q.device
    cells = (batch, desc.num_q_heads)
    out = torch.empty(batch, desc.num_q_heads, desc.head_dim, dtype=torch.float32, device=dev) if out is None else out
    meter = torch.empty(cells, dtype=torch.float32, device=dev) if meter is None else meter
    meter_raw = torch.empty(cells, dtype=torch.float32, device=dev) if meter_raw is None else meter_raw
    meter_b = torch.empty(cells, dtype=torch.float32, device=dev) if meter_b is None else meter_b
    meter_b_raw = torch.empty(cells, dtype=torch.float32, device=dev) if meter_b_raw is None else meter_b_raw
    d = desc.c()
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        _decode_g32(d, layer, q, block_table, ctx_lens, cache, ws, delta_loc, out, meter, meter_raw, meter_b,
                    meter_b_raw, stream)
        return out, meter, meter_raw, meter_b, meter_b_raw
    _check(lib.wc_metered_decode_attention_tier_b(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), float(delta_loc), _ptr(out), _ptr(meter), _ptr(meter_raw), _ptr(meter_b),
        _ptr(meter_b_raw), ws.ptr(), ws.nbytes, _stream(stream)))
    return out, meter, meter_raw, meter_b, meter_b_raw


def metered_decode_attention_v(desc: CacheDesc, layer: int, q: torch.Tensor, block_table: torch.Tensor,
                               ctx_lens: torch.Tensor, cache: LayerCache, ws: Workspace, out=None, meter=None,
                               meter_raw=None, value_term=None, v_max=None, out_bound=None, stream=None):
    """``wc_metered_decode_attention_v``; returns (out, meter, meter_raw, value_term, v_max, out_bound)."""
    if cache.v_witness is None:
        raise ValueError("the cache holds no value witness (LayerCache.empty(..., value_witness=True))")
    batch, max_pages = block_table.shape
    dev = q.device
    cells = (batch, desc.num_q_heads)
    new = lambda t: torch.empty(cells, dtype=torch.float32, device=dev) if t is None else t
    out = torch.empty(batch, desc.num_q_heads, desc.head_dim, dtype=torch.float32, device=dev) if out is None else out
    meter, meter_raw, value_term, v_max, out_bound = map(new, (meter, meter_raw, value_term, v_max, out_bound))
    d = desc.c()
    _check(lib.wc_metered_decode_attention_v(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), _ptr(cache.v_witness), _ptr(out), _ptr(meter), _ptr(meter_raw),
        _ptr(value_term), _ptr(v_max), _ptr(out_bound), ws.ptr(), ws.nbytes, _stream(stream)))
    return out, meter, meter_raw, value_term, v_max, out_bound


def metered_decode_attention_repair(desc: CacheDesc, layer: int, q: torch.Tensor, block_table: torch.Tensor,
                                    ctx_lens: torch.Tensor, cache: LayerCache, ws: Workspace, out=None, meter=None,
                                    meter_raw=None, page_terms=None, softmax_norm=None, stream=None):
    """``wc_metered_decode_attention_repair``; returns (out, meter, meter_raw, page_terms [B,Hq,max_pages,2],
    softmax_norm [B,Hq,2])."""
    batch, max_pages = block_table.shape
    dev = q.device
    cells = (batch, desc.num_q_heads)
    out = torch.empty(batch, desc.num_q_heads, desc.head_dim, dtype=torch.float32, device=dev) if out is None else out
    meter = torch.empty(cells, dtype=torch.float32, device=dev) if meter is None else meter
    meter_raw = torch.empty(cells, dtype=torch.float32, device=dev) if meter_raw is None else meter_raw
    if page_terms is None:
        page_terms = torch.empty(batch, desc.num_q_heads, max_pages, 2, dtype=torch.float32, device=dev)
    if softmax_norm is None:
        softmax_norm = torch.empty(batch, desc.num_q_heads, 2, dtype=torch.float32, device=dev)
    d = desc.c()
    _check(lib.wc_metered_decode_attention_repair(
        ctypes.byref(d), layer, _ptr(q), _ptr(block_table), max_pages, _ptr(ctx_lens), batch,
        _ptr(cache.k_codes), _ptr(cache.v_codes), _ptr(cache.k_scale), _ptr(cache.v_scale),
        _ptr(cache.k_witness), _ptr(out), _ptr(meter), _ptr(meter_raw), _ptr(page_terms), _ptr(softmax_norm),
        ws.ptr(), ws.nbytes, _stream(stream)))
    return out, meter, meter_raw, page_terms, softmax_norm


def repair_select(page_terms: torch.Tensor, softmax_norm: torch.Tensor, ctx_lens: torch.Tensor, tau: float,
                  keep_q=None, contrib=True, repair_pages=None, n_repair=None, d_after=None, dev_status=None,
                  stream=None):
    """``wc_repair_select``; returns (contrib [B,Hq,max_pages] fp32 or None, repair_pages int32
    [B,Hq,max_pages] (the first n_repair entries of a row are meaningful), n_repair int32 [B,Hq],
    d_after fp32 [B,Hq]).  ``contrib=False`` skips storing the contributions."""
    batch, num_q_heads, max_pages = page_terms.shape[:3]
    dev = page_terms.device
    if contrib is True:
        contrib = torch.zeros(batch, num_q_heads, max_pages, dtype=torch.float32, device=dev)
    elif contrib is False:
        contrib = None
    if repair_pages is None:
        repair_pages = torch.full((batch, num_q_heads, max_pages), -1, dtype=torch.int32, device=dev)
    n_repair = torch.empty(batch, num_q_heads, dtype=torch.int32, device=dev) if n_repair is None else n_repair
    d_after = torch.empty(batch, num_q_heads, dtype=torch.float32, device=dev) if d_after is None else d_after
    _check(lib.wc_repair_select(_ptr(page_terms), _ptr(softmax_norm), _ptr(ctx_lens), batch, num_q_heads, max_pages,
                                _ptr(keep_q), float(tau), _ptr(contrib), _ptr(repair_pages), _ptr(n_repair),
                                _ptr(d_after), _ptr(dev_status), _stream(stream)))
    return contrib, repair_pages, n_repair, d_after


def gate_joint(meter_raw: torch.Tensor, value_term: torch.Tensor, v_max: torch.Tensor, group: int, tau_k: float,
               tau_v: float, keep_q=None, keep_kv=None, n_kept=None, stream=None):
    """``wc_gate_joint``: returns (keep_q uint8 [n], keep_kv uint8 [n/group], n_kept int32 [2])."""
    n = meter_raw.numel()
    dev = meter_raw.device
    keep_q = torch.empty(n, dtype=torch.uint8, device=dev) if keep_q is None else keep_q
    keep_kv = torch.empty(n // group, dtype=torch.uint8, device=dev) if keep_kv is None else keep_kv
    n_kept = torch.empty(2, dtype=torch.int32, device=dev) if n_kept is None else n_kept
    _check(lib.wc_gate_joint(_ptr(meter_raw), _ptr(value_term), _ptr(v_max), n, group, float(tau_k), float(tau_v),
                             _ptr(keep_q), _ptr(keep_kv), _ptr(n_kept), _stream(stream)))
    return keep_q, keep_kv, n_kept


def gate(meter_raw: torch.Tensor, group: int, tau: float, keep_q=None, keep_kv=None, n_kept=None,
         stream=None):
    """``wc_gate``: returns (keep_q uint8 [n], keep_kv uint8 [n/group], n_kept int32 [2])."""
    n = meter_raw.numel()
    dev = meter_raw.device
    keep_q = torch.empty(n, dtype=torch.uint8, device=dev) if keep_q is None else keep_q
    keep_kv = torch.empty(n // group, dtype=torch.uint8, device=dev) if keep_kv is None else keep_kv
    n_kept = torch.empty(2, dtype=torch.int32, device=dev) if n_kept is None else n_kept
    _check(lib.wc_gate(_ptr(meter_raw), n, group, float(tau), _ptr(keep_q), _ptr(keep_kv),
                       _ptr(n_kept), _stream(stream)))
    return keep_q, keep_kv, n_kept


def read_status(ws_or_word, stream=None) -> int:
    """Synchronising read-and-clear of the device status word; returns the bits."""
    if isinstance(ws_or_word, Workspace):
        p, is_word = ws_or_word.ptr(), 0
    else:
        p, is_word = _ptr(ws_or_word), 1
    bits = ctypes.c_uint32(0)
    st = lib.wc_read_status(p, is_word, ctypes.byref(bits), _stream(stream))
    if st not in (0, 5):
        _check(st)
    return bits.value


def version():
    v = lib.wc_version()
    return (v >> 16, v & 0xFFFF)
