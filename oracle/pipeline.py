"""The write path over a paged cache and one metered decode step.

Test infrastructure only (see ``oracle/__init__.py``).

Paged cache (PagedAttention-style token slots, §6.2.3; 16-token pages as in
the serving runs of §6.2 and Table "serving"): slot = page * P + offset with
P = page_size; per layer the arrays are

  k_codes, v_codes  [num_pages, Hkv, P, d]   int8 (dither) or uint8 (fp8 bytes)
  k_scale, v_scale  [num_pages, Hkv, P]      fp16 (dither scheme only)
  k_witness         [num_pages, Hkv, P, B]   fp16

and for the grouped scheme (§6.2.3) k_scale, v_scale [num_pages, Hkv, P, d/G_c]
(one per channel group), k_bypass [num_pages, Hkv, P, 2m] fp16 (the exact
values of the m bypassed RoPE pairs, pair by pair) and bypass_pairs [Hkv, m],
the layer's fixed pair set per KV head.

Reading (storage order, grouped scheme): the paper fixes neither the byte
order of a stored row nor which dither word serves which channel.  The
grouped scheme stores a row's channels in a fixed permuted order and draws
the dither by storage position (byte i of the Philox call with channel-group
index n serves storage position 16 n + i, the same rule as the per-token
scheme's identity order).  Storage position p holds channel
  K:  16 ((p >> 2) & 7) + 4 (p >> 5) + (p & 3)
  V:  16 ((p >> 1) & 7) + 8 (p & 1) + (p >> 4)
(the order in which the decode's matrix-multiply fragments consume them, so
that each fragment step meets one channel group).

The meter loop (§6 box): write path quantizes k -> k^ and stores the
witness; the read path computes the compressed attention and
A = sum_t p~_t e^{c_t}; meter = min(1, 1/2 (A^2 - 1)); the gate compares it
with tau.  The query head h_q reads KV head h_q // G (grouped-query
attention, G = Hq / Hkv).
"""

from dataclasses import dataclass

import numpy as np

from . import meter as M
from . import fp, philox, quantizer

SCHEME_DITHER_INT8 = 0
SCHEME_FP8_E4M3 = 1
SCHEME_DITHER_INT8_G32 = 2     # grouped scales + fixed-channel outlier bypass (§6.2.3)


@dataclass
class Desc:
    head_dim: int = 128
    num_q_heads: int = 8
    num_kv_heads: int = 2
    num_bands: int = 8
    page_size: int = 16
    num_pages: int = 256
    scheme: int = SCHEME_DITHER_INT8
    rope_layout: int = quantizer.ROPE_HALF
    dither_bits: int = 8
    seed: int = 0
    group_channels: int = 32      # G_c, grouped scheme
    num_bypass_pairs: int = 0     # m, grouped scheme


def empty_cache(desc):
    shp = (desc.num_pages, desc.num_kv_heads, desc.page_size)
    code_t = np.uint8 if desc.scheme == SCHEME_FP8_E4M3 else np.int8
    cache = {
        "k_codes": np.zeros(shp + (desc.head_dim,), code_t),
        "v_codes": np.zeros(shp + (desc.head_dim,), code_t),
        "k_witness": np.zeros(shp + (desc.num_bands,), np.float16),
        "v_witness": np.zeros(shp + (2,), np.float16),       # (rho^v, ||v||), rounded up
    }
    if desc.scheme == SCHEME_DITHER_INT8:
        cache["k_scale"] = np.zeros(shp, np.float16)
        cache["v_scale"] = np.zeros(shp, np.float16)
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        ng = desc.head_dim // desc.group_channels
        cache["k_scale"] = np.zeros(shp + (ng,), np.float16)
        cache["v_scale"] = np.zeros(shp + (ng,), np.float16)
        cache["k_bypass"] = np.zeros(shp + (2 * desc.num_bypass_pairs,), np.float16)
        cache["bypass_pairs"] = np.zeros((desc.num_kv_heads, desc.num_bypass_pairs), np.int64)
    return cache


def storage_order(head_dim, tag):
    """Channel held by each storage position of a grouped-scheme row (K: tag 0, V: tag 1)."""
    p = np.arange(head_dim)
    if tag == 0:
        return 16 * ((p >> 2) & 7) + 4 * (p >> 5) + (p & 3)
    return 16 * ((p >> 1) & 7) + 8 * (p & 1) + (p >> 4)


def _grouped_dither(desc, layer, kv_head, slots, tag):
    """xi [n, d] by channel: the storage-position dither moved to its channels."""
    xi_pos = philox.dither_values(philox.dither_integers(
        desc.seed, layer, kv_head, slots, tag, desc.head_dim, desc.dither_bits), desc.dither_bits)
    xi = np.empty_like(xi_pos)
    xi[:, storage_order(desc.head_dim, tag)] = xi_pos
    return xi


def _excluded(desc, cache, kv_head, tag):
    """Bypassed dims of a KV head: keys only (tag 0)."""
    if tag != 0 or desc.num_bypass_pairs == 0:
        return np.zeros(0, np.int64)
    return quantizer.bypass_dims(cache["bypass_pairs"][kv_head], desc.head_dim, desc.rope_layout)


def quantize_rows(desc, layer, kv_head, rows16, slots, tag, excluded=()):
    """Quantize fp16 rows [n, d] written to ``slots``.

    Returns (codes by channel, scale or None, reconstruction float64 [n, d]);
    ``excluded`` are the bypassed dims of the grouped scheme (exact, code 0).
    """
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        G = desc.group_channels
        s = quantizer.group_scales(rows16, G, excluded)
        s_chan = np.repeat(s, G, axis=-1)
        xi = _grouped_dither(desc, layer, kv_head, slots, tag)
        code = quantizer.dither_code(rows16, s_chan, xi)
        rec = quantizer.dither_reconstruct(code, s_chan, xi)
        if len(excluded):
            code[:, excluded] = 0
            rec[:, excluded] = np.asarray(rows16, dtype=np.float16)[:, excluded].astype(np.float64)
        return code, s, rec
    if desc.scheme == SCHEME_DITHER_INT8:
        s = quantizer.int8_scale(rows16)
        j = philox.dither_integers(desc.seed, layer, kv_head, slots, tag,
                                   desc.head_dim, desc.dither_bits)
        xi = philox.dither_values(j, desc.dither_bits)
        code = quantizer.dither_code(rows16, s, xi)
        return code, s, quantizer.dither_reconstruct(code, s, xi)
    code, rec = quantizer.fp8_quantize(rows16)
    return code, None, rec


def write_tokens(desc, layer, k16, v16, slot_mapping, cache, bypass_pairs=None):
    """kv_quantize_witness: k16, v16 [n_tok, Hkv, d] fp16; slot < 0 skips.

    Grouped scheme: ``bypass_pairs`` [Hkv, m] is the layer's fixed pair set
    (kept in the cache for the read side).
    """
    if desc.scheme == SCHEME_DITHER_INT8_G32 and desc.num_bypass_pairs:
        cache["bypass_pairs"][...] = np.asarray(bypass_pairs, dtype=np.int64).reshape(
            desc.num_kv_heads, desc.num_bypass_pairs)
    slot_mapping = np.asarray(slot_mapping, dtype=np.int64)
    live = slot_mapping >= 0
    slots = slot_mapping[live]
    page, off = slots // desc.page_size, slots % desc.page_size
    for h in range(desc.num_kv_heads):
        kr = np.asarray(k16)[live, h, :]
        vr = np.asarray(v16)[live, h, :]
        excl = _excluded(desc, cache, h, 0) if desc.scheme == SCHEME_DITHER_INT8_G32 else ()
        kc, ks, khat = quantize_rows(desc, layer, h, kr, slots, 0, excl)
        vc, vs, vhat = quantize_rows(desc, layer, h, vr, slots, 1)
        if len(excl):
            cache["k_bypass"][page, h, off] = kr[:, excl]
        if desc.scheme == SCHEME_DITHER_INT8_G32:     # storage order
            kc, vc = kc[:, storage_order(desc.head_dim, 0)], vc[:, storage_order(desc.head_dim, 1)]
        cache["k_codes"][page, h, off] = kc
        cache["v_codes"][page, h, off] = vc
        if ks is not None:
            cache["k_scale"][page, h, off] = ks
            cache["v_scale"][page, h, off] = vs
        resid = khat - kr.astype(np.float64)
        cache["k_witness"][page, h, off] = quantizer.witness(
            resid, desc.num_bands, desc.rope_layout)
        cache["v_witness"][page, h, off] = quantizer.value_witness(vhat - vr.astype(np.float64), vr)


def slots_of(desc, block_table_row, ctx_len):
    t = np.arange(ctx_len)
    return np.asarray(block_table_row)[t // desc.page_size] * desc.page_size + t % desc.page_size


def reconstruct(desc, layer, kv_head, slots, cache):
    """Dequantized k^, v^ [S, d] float64 and the stored witness [S, B]."""
    page, off = slots // desc.page_size, slots % desc.page_size
    kc = cache["k_codes"][page, kv_head, off]
    vc = cache["v_codes"][page, kv_head, off]
    if desc.scheme == SCHEME_DITHER_INT8_G32:
        G = desc.group_channels
        xk = _grouped_dither(desc, layer, kv_head, slots, 0)
        xv = _grouped_dither(desc, layer, kv_head, slots, 1)
        kc, vc = np.empty_like(kc), np.empty_like(vc)              # back to channel order
        kc[:, storage_order(desc.head_dim, 0)] = cache["k_codes"][page, kv_head, off]
        vc[:, storage_order(desc.head_dim, 1)] = cache["v_codes"][page, kv_head, off]
        khat = quantizer.dither_reconstruct(kc, np.repeat(cache["k_scale"][page, kv_head, off], G, axis=-1), xk)
        vhat = quantizer.dither_reconstruct(vc, np.repeat(cache["v_scale"][page, kv_head, off], G, axis=-1), xv)
        excl = _excluded(desc, cache, kv_head, 0)
        if len(excl):
            khat[:, excl] = cache["k_bypass"][page, kv_head, off].astype(np.float64)
    elif desc.scheme == SCHEME_DITHER_INT8:
        xk = philox.dither_values(philox.dither_integers(
            desc.seed, layer, kv_head, slots, 0, desc.head_dim, desc.dither_bits), desc.dither_bits)
        xv = philox.dither_values(philox.dither_integers(
            desc.seed, layer, kv_head, slots, 1, desc.head_dim, desc.dither_bits), desc.dither_bits)
        khat = quantizer.dither_reconstruct(kc, cache["k_scale"][page, kv_head, off], xk)
        vhat = quantizer.dither_reconstruct(vc, cache["v_scale"][page, kv_head, off], xv)
    else:
        khat, vhat = fp.e4m3_decode(kc), fp.e4m3_decode(vc)
    return khat, vhat, cache["k_witness"][page, kv_head, off]


def decode_sequence(desc, layer, q16, block_table_row, ctx_len, cache,
                    k_exact=None, v_exact=None, delta_loc=None, repair_tau=None):
    """metered_decode_attention for one sequence: q16 [Hq, d] post-RoPE.

    Returns a dict with float64 ``out`` [Hq, d], ``meter``/``meter_raw``
    [Hq]; with the exact fp16 keys/values [S, Hkv, d] also ``tv`` [Hq]
    (the true TV between exact and compressed attention) and
    ``out_exact`` [Hq, d]; with ``delta_loc`` (dithered INT8 only) also the
    Tier-B meters ``meter_b``/``meter_b_raw`` [Hq] (§4.2); with ``repair_tau``
    also ``contrib`` [Hq, pages] (page contributions to D) and ``repair``
    (per query head: the logical pages to page in, in order, §6.3.5).
    """
    G = desc.num_q_heads // desc.num_kv_heads
    d = desc.head_dim
    slots = slots_of(desc, block_table_row, ctx_len)
    res = {k: np.zeros((desc.num_q_heads, d)) for k in ("out", "out_exact")}
    for k in ("meter", "meter_raw", "tv", "A", "meter_b", "meter_b_raw", "value_term", "v_max", "out_bound",
              "out_err"):
        res[k] = np.zeros(desc.num_q_heads)
    tier_b = delta_loc is not None
    n_pages = (ctx_len + desc.page_size - 1) // desc.page_size
    if repair_tau is not None:
        res["contrib"] = np.zeros((desc.num_q_heads, n_pages))
        res["repair"] = [None] * desc.num_q_heads
    if tier_b and desc.scheme == SCHEME_FP8_E4M3:
        raise ValueError("Tier B needs the dithered INT8 cache (a controlled quantizer)")
    if ctx_len == 0:
        # An empty context attends to nothing: out = 0 and meter = meter_raw = 0
        # (A = 1 in the e-form), no pages to repair (the reading used for context 0).
        res["A"][:] = 1.0
        if repair_tau is not None:
            res["repair"] = [np.zeros(0, dtype=np.int64) for _ in range(desc.num_q_heads)]
        return res
    page, off = slots // desc.page_size, slots % desc.page_size
    for h in range(desc.num_kv_heads):
        khat, vhat, w = reconstruct(desc, layer, h, slots, cache)
        for g in range(G):
            hq = h * G + g
            q = np.asarray(q16[hq], dtype=np.float64)
            z_tilde = M.logits(q, khat)
            c = M.tier_a_bound(q, w, desc.num_bands, desc.rope_layout)
            p_tilde, terms = M.eform_terms(z_tilde, c)
            res["meter"][hq], res["meter_raw"][hq], res["A"][hq] = M.meter_of_terms(terms)
            res["out"][hq] = M.attend(p_tilde, vhat)
            if repair_tau is not None:
                res["contrib"][hq] = M.page_contributions(p_tilde, c, np.arange(ctx_len) // desc.page_size, n_pages,
                                                          terms=terms)
                res["repair"][hq] = M.repair_plan(res["contrib"][hq], repair_tau)[0]
            vw = cache["v_witness"][page, h, off].astype(np.float64)        # [S, 2]
            res["value_term"][hq] = M.value_term(p_tilde, vw[:, 0])
            res["v_max"][hq] = np.max(vw[:, 1]) if ctx_len else 0.0
            res["out_bound"][hq] = M.output_bound(res["meter"][hq], res["v_max"][hq], res["value_term"][hq])
            if tier_b and desc.scheme == SCHEME_DITHER_INT8_G32:
                u = M.tier_b_bound_grouped(q, cache["k_scale"][page, h, off], desc.group_channels,
                                           _excluded(desc, cache, h, 0), ctx_len, delta_loc)
                res["meter_b"][hq], res["meter_b_raw"][hq], _ = M.eform_meter_logits(z_tilde, u)
            elif tier_b:
                u = M.tier_b_bound(q, cache["k_scale"][page, h, off].astype(np.float64), ctx_len, delta_loc)
                res["meter_b"][hq], res["meter_b_raw"][hq], _ = M.eform_meter_logits(z_tilde, u)
            if k_exact is not None:
                p = M.softmax(M.logits(q, np.asarray(k_exact)[:ctx_len, h]))
                res["tv"][hq] = M.total_variation(p, p_tilde)
                res["out_exact"][hq] = M.attend(p, np.asarray(v_exact)[:ctx_len, h])
                res["out_err"][hq] = np.linalg.norm(res["out_exact"][hq] - res["out"][hq])
    return res
