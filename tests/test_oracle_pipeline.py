"""End-to-end pins for oracle.pipeline: soundness of the meter against the
true TV on quantized caches (random and adversarial queries), GQA head
mapping, paging invariance (no GPU)."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as M
from oracle import quantizer as Q
from oracle.pipeline import Desc, decode_sequence, empty_cache, reconstruct, slots_of, write_tokens


def _small(scheme, seed=0, ctx=300, shuffle=True, bits=8, layout=Q.ROPE_HALF):
    wl = W.Workload("t", 1, 8, 2, [ctx, ctx // 2 + 7], scheme=scheme, shuffle_pages=shuffle, seed=seed)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, 0)
    q = W.layer_queries(wl, 0)
    desc = Desc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=scheme,
                dither_bits=bits, rope_layout=layout, seed=seed + 11)
    cache = empty_cache(desc)
    write_tokens(desc, 0, k.numpy(), v.numpy(), sm, cache)
    return wl, bt, k.numpy(), v.numpy(), q.numpy(), desc, cache


@pytest.mark.parametrize("scheme,bits", [(0, 8), (0, 10), (1, 8)])
def test_meter_bounds_true_tv(scheme, bits):
    wl, bt, k, v, q, desc, cache = _small(scheme, bits=bits)
    off = 0
    for b, S in enumerate(wl.ctx_lens):
        r = decode_sequence(desc, 0, q[b], bt[b], S, cache, k[off:off + S], v[off:off + S])
        assert np.all(r["tv"] > 0)
        assert np.all(r["tv"] <= r["meter_raw"])
        assert np.all(r["meter"] <= 1.0)
        off += S


def test_meter_bounds_tv_for_adversarial_queries():
    """Queries aligned band by band with one token's residual make that
    token's Cauchy-Schwarz step tight; the meter must still bound TV."""
    wl, bt, k, v, q, desc, cache = _small(0, ctx=200, shuffle=False)
    S = wl.ctx_lens[0]
    slots = slots_of(desc, bt[0], S)
    khat, vhat, w = reconstruct(desc, 0, 0, slots, cache)
    resid = khat - k[:S, 0].astype(np.float64)
    dims = Q.band_dims(128, 8, Q.ROPE_HALF)
    rng = np.random.default_rng(30)
    for t in [0, 1, 57, S - 1]:
        for scale in [1.0, 30.0, 300.0]:
            qa = np.zeros(128)
            for b in range(8):
                qa[dims[b]] = rng.uniform(0.5, 1.5) * resid[t, dims[b]]
            qa = qa / np.linalg.norm(qa) * scale
            q16 = np.tile(qa.astype(np.float16), (8, 1))
            r = decode_sequence(desc, 0, q16, bt[0], S, cache, k[:S], v[:S])
            assert np.all(r["tv"] <= r["meter_raw"])
            # logit error of token t is (nearly) at its bound
            c = M.tier_a_bound(q16[0].astype(np.float64), w, 8, Q.ROPE_HALF)
            eps = resid @ q16[0].astype(np.float64) / np.sqrt(128)
            assert abs(eps[t]) >= 0.98 * c[t]
            assert np.all(np.abs(eps) <= c * (1 + 1e-12))


def test_gqa_head_mapping_and_paging_invariance():
    """Query head h reads KV head h // G, and shuffling the physical pages
    changes no decode result (the dither is keyed by slot, so the codes
    move with the slot but the reconstruction is the same)."""
    wl, bt, k, v, q, desc, cache = _small(1, shuffle=True)
    wl2, bt2, _, _, _, desc2, cache2 = _small(1, shuffle=False)
    S = wl.ctx_lens[0]
    r1 = decode_sequence(desc, 0, q[0], bt[0], S, cache)
    r2 = decode_sequence(desc2, 0, q[0], bt2[0], S, cache2)
    assert np.allclose(r1["out"], r2["out"], rtol=1e-12) and np.allclose(r1["meter_raw"], r2["meter_raw"], rtol=1e-12)
    # swap the two KV heads' data: the two query-head groups swap results
    q_sw = np.concatenate([q[0][4:], q[0][:4]])
    cache_sw = {name: arr[:, ::-1].copy() for name, arr in cache.items()}
    r3 = decode_sequence(desc, 0, q_sw, bt[0], S, cache_sw)
    assert np.allclose(r3["out"][:4], r1["out"][4:], rtol=1e-12)
    assert np.allclose(r3["meter_raw"][4:], r1["meter_raw"][:4], rtol=1e-12)


def test_write_path_is_position_free_and_deterministic():
    wl, bt, k, v, q, desc, cache = _small(0)
    _, _, _, _, _, _, cache_b = _small(0)
    for name in cache:
        assert np.array_equal(cache[name].view(np.uint8), cache_b[name].view(np.uint8))
    # skipped slots (-1) leave the cache untouched
    c2 = empty_cache(desc)
    write_tokens(desc, 0, k[:5], v[:5], np.array([-1, 3, -1, 4, -1]), c2)
    assert np.count_nonzero(c2["k_codes"][0, :, [0, 1, 2, 5]]) == 0
    assert np.count_nonzero(c2["k_codes"][0, :, 3]) > 0


@pytest.mark.parametrize("scheme", [0, 1])
def test_empty_context_attends_to_nothing(scheme):
    """Context 0 (the reading for an empty sequence): out = 0, meters 0, no
    pages to repair; a one-token context next to it is an ordinary decode."""
    wl, bt, k, v, q, desc, cache = _small(scheme)
    r0 = decode_sequence(desc, 0, q[0], bt[0], 0, cache, k[:0], v[:0], repair_tau=0.1,
                         delta_loc=1e-3 if scheme == 0 else None)
    for name in ("out", "meter", "meter_raw", "tv", "value_term", "out_bound", "meter_b_raw"):
        assert np.all(r0[name] == 0), name
    assert all(len(x) == 0 for x in r0["repair"])
    r1 = decode_sequence(desc, 0, q[0], bt[0], 1, cache, k[:1], v[:1])
    assert np.all(r1["meter_raw"] >= r1["tv"])
    assert np.allclose(np.abs(r1["out"]).sum(axis=1) > 0, True)
