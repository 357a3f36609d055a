"""Pins for the oracle's value-side witness and output bound (§3, §4.2):
soundness of ||y - y^|| <= 2 TV max||v|| + sum p~ rho^v against the exact
output, tightness when the key error vanishes and the value residuals are
parallel, the stored witness rounding, the fp8 case with exactly
representable values, and the joint gate's decisions."""

import numpy as np
import pytest

import workloads as W
from oracle import fp
from oracle import meter as M
from oracle import pipeline as OP
from oracle import quantizer as Q


@pytest.mark.parametrize("scheme", [OP.SCHEME_DITHER_INT8, OP.SCHEME_FP8_E4M3])
def test_output_bound_is_sound(scheme):
    wl = W.Workload("v", 1, 8, 2, [300, 57], shuffle_pages=True, seed=3)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, 0)
    q = W.layer_queries(wl, 0).numpy()
    od = OP.Desc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=scheme, seed=9)
    cache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k.numpy(), v.numpy(), sm, cache)
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    for b, S in enumerate(wl.ctx_lens):
        for scale in (1.0, 4.0, 16.0):                 # concentrated attention as well
            r = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S, cache,
                                   k.numpy()[offs[b]:offs[b] + S], v.numpy()[offs[b]:offs[b] + S])
            assert np.all(r["out_err"] <= r["out_bound"] * (1 + 1e-12))
            assert np.all(r["value_term"] > 0)


def test_bound_tight_for_parallel_residuals_without_key_error():
    rng = np.random.default_rng(0)
    S, d = 50, 128
    p_t = M.softmax(rng.standard_normal(S))
    e = rng.standard_normal(d); e /= np.linalg.norm(e)
    rho = rng.uniform(0.01, 0.2, S)
    v = rng.standard_normal((S, d))
    vhat = v + rho[:, None] * e                      # all residuals along e
    err = np.linalg.norm(M.attend(p_t, v) - M.attend(p_t, vhat))
    bound = M.output_bound(0.0, np.max(np.linalg.norm(v, axis=1)), M.value_term(p_t, rho))
    assert err == pytest.approx(bound, rel=1e-12)    # the triangle inequality is attained


def test_value_witness_rounds_up_by_at_most_one_ulp():
    rng = np.random.default_rng(1)
    r = rng.standard_normal((200, 128)) * rng.lognormal(-4, 1, (200, 1))
    v = rng.standard_normal((200, 128))
    w = Q.value_witness(r, v).astype(np.float64)
    exact = np.stack([np.linalg.norm(r, axis=1), np.linalg.norm(v, axis=1)], axis=1)
    assert np.all(w >= exact)
    below = (Q.value_witness(r, v).view(np.uint16) - 1).view(np.float16).astype(np.float64)
    assert np.all(below < exact)                     # the next fp16 down is already too small


def test_fp8_values_exactly_representable_give_zero_value_error():
    vals = fp.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))    # positive finite e4m3 values
    v16 = np.resize(vals, (3, 1, 128)).astype(np.float16)
    od = OP.Desc(num_q_heads=1, num_kv_heads=1, num_pages=1, scheme=OP.SCHEME_FP8_E4M3)
    cache = OP.empty_cache(od)
    OP.write_tokens(od, 0, v16, v16, np.array([0, 1, 2]), cache)
    assert np.all(cache["v_witness"][0, 0, :3, 0] == 0)


def test_joint_gate_decisions():
    mr = np.array([0.1, 0.1, 0.05, np.nan, 0.0, 0.2], np.float32)
    vt = np.array([0.5, 0.51, 0.0, 0.0, np.inf, 0.0], np.float32)
    vm = np.array([5.0, 5.0, 1.0, 1.0, 1.0, 1.0], np.float32)
    keep_q, keep_kv, nq, nkv = M.joint_gate(mr, vt, vm, 0.1, 0.1, 2)
    assert keep_q.tolist() == [True, False, True, False, False, False]   # equality keeps, NaN / inf fall back
    assert keep_kv.tolist() == [False, False, False] and (nq, nkv) == (2, 0)
