"""The meter when one token's bound is huge and its softmax weight is not
representable in fp32 (§3 Thm. "Sound replacement": the meter stays an upper
bound, +inf standing for overflow).

A key row of magnitude A (its scale, and with it the residual witness, grows
with A) gets a Tier-A bound c with cl = c log2(e) near a target; an anchor token
on the same page (so the same warp's running maximum), a flat row signed like the
first query, sets the maximum, so that the huge token's weight 2^t in the log2 frame of
the maximum sits near a target t below -126, where fp32 (flushed) holds 0.  The
token's term p~ (e^c - 1) = 2^t (2^cl - 1) is still about 2^(t + cl):

  * "finite": cl ~ 125, t ~ -130: a term of ~2^-5, a sizeable part of D, which a
    product 0 * (2^cl - 1) drops (a meter below the exact one);
  * "large":  cl ~ 200, t ~ -150: a term of ~2^50 (2^cl is beyond fp32, so the
    product is 0 * inf = NaN);
  * "small":  cl ~ 200, t ~ -250: a term of ~2^-50.

The GPU's meters must match the oracle's (after rounding to fp32, where
overflow is +inf), lie on or above them, and never be NaN."""

import numpy as np
import pytest
import torch

import workloads as W
from oracle import meter as OM
from oracle import pipeline as OP
from tests._parity import assert_close, assert_sound, make_inputs, numpy_cache_to_gpu

LOG2E = 1.4426950408889634
S, J, ANCHOR = 40, 21, 20          # both on logical page 1 (tokens 16-31)
CASES = {"finite": (125.0, -130.0), "large": (200.0, -150.0), "small": (200.0, -250.0)}
DELTA_LOC = 0.01


def build_case(scheme, bits, case):
    """CPU inputs and the oracle's cache for one case (the oracle only)."""
    cl_target, t_target = CASES[case]
    wl = W.Workload("extreme", 1, 4, 1, [S], scheme=scheme, shuffle_pages=True, seed=31)
    bt, sm, k, v, q = make_inputs(wl, 0)
    od = OP.Desc(num_q_heads=4, num_kv_heads=1, num_pages=wl.num_pages, scheme=scheme, dither_bits=bits, seed=9)
    slots = OP.slots_of(od, bt[0], S)
    q16 = q.numpy()
    q0 = q16[0, 0].astype(np.float64)
    qhat = q0 / np.linalg.norm(q0)
    sgn = np.sign(q0)                                       # the anchor: gamma * sign(q0), one scale for
    scale = np.abs(q0).sum() / np.sqrt(q0.size) * LOG2E     # the largest logit per unit of bound
    vv = v.numpy()
    for useed in range(40):
        rng = np.random.default_rng(1000 + useed)
        u = rng.choice([-1.0, 1.0], 128) * rng.uniform(0.5, 1.0, 128)
        u -= (u @ qhat) * qhat                 # no logit of its own: only its quantization moves it
        kk = k.numpy().copy()

        def at(a, gamma):
            kk[J, 0] = (a * u).astype(np.float16)
            kk[ANCHOR, 0] = (gamma * sgn).astype(np.float16)
            cache = OP.empty_cache(od)
            OP.write_tokens(od, 0, kk, vv, sm, cache)
            khat, _, w = OP.reconstruct(od, 0, 0, slots, cache)
            return cache, OM.logits(q0, khat) * LOG2E, OM.tier_a_bound(q0, w, od.num_bands, od.rope_layout) * LOG2E

        lo, hi = 0.0, np.log(60000.0)          # the huge row's magnitude: bisection on its bound
        for _ in range(36):
            mid = 0.5 * (lo + hi)
            if at(np.exp(mid), 0.0)[2][J] < cl_target:
                lo = mid
            else:
                hi = mid
        a = float(np.exp(hi))
        _, y, cl = at(a, 0.0)
        others = np.delete(y, [J, ANCHOR])
        want = y[J] - t_target                 # the anchor's logit that puts t at its target
        if want < others.max() + 4.0:          # the anchor must stay the maximum
            continue
        gamma = want / scale
        for _ in range(3):                     # its quantization moves its logit a little
            cache, y, cl = at(a, gamma)
            gamma += (want - y[ANCHOR]) / scale
        cache, y, cl = at(a, gamma)
        if np.max(np.abs(kk[ANCHOR, 0].astype(np.float64))) > 60000:
            continue
        t = y[J] - y.max()
        if int(np.argmax(y)) == ANCHOR and abs(t - t_target) < 3.0:
            return dict(wl=wl, bt=bt, q16=q16, k=kk, v=vv, od=od, cache=cache, t=t, cl=cl[J])
    raise AssertionError(f"no input lands in case {case}")


def _regime_checks(case, t, cl):
    cl_target, t_target = CASES[case]
    assert t <= -127.0, "the huge token's weight must underflow fp32"
    if case == "finite":
        assert 106.0 < cl < 128.0 and t + cl > -10.0, (t, cl)    # 2^cl finite, the term far from 0
    else:
        assert cl >= 140.0, cl                                    # 2^cl beyond fp32
        if case == "large":
            assert 40.0 < t + cl < 80.0, (t, cl)
        else:
            assert t + cl < -20.0, (t, cl)


SCHEMES = [(0, 8), (0, 10), (2, 8), (1, 8)]
PARAMS = [(s, b, c) for s, b in SCHEMES for c in CASES if s != 1 or c != "finite"]


@pytest.mark.parametrize("scheme,bits,case", PARAMS)
def test_extreme_inputs_land_in_their_regime(scheme, bits, case):
    """The constructed inputs reach the regime they are meant for (oracle only),
    and in the "finite" case dropping the token's term would move the meter far
    beyond the parity tolerance."""
    c = build_case(scheme, bits, case)
    _regime_checks(case, c["t"], c["cl"])
    r = OP.decode_sequence(c["od"], 0, c["q16"][0], c["bt"][0], S, c["cache"])
    assert np.isfinite(r["meter_raw"][0]) or case != "finite"
    if case == "finite":
        khat, _, w = OP.reconstruct(c["od"], 0, 0, OP.slots_of(c["od"], c["bt"][0], S), c["cache"])
        q0 = c["q16"][0, 0].astype(np.float64)
        p = OM.softmax(OM.logits(q0, khat))
        cb = OM.tier_a_bound(q0, w, c["od"].num_bands, c["od"].rope_layout)
        p_drop = p.copy()
        p_drop[J] = 0.0
        full, dropped = OM.eform_meter(p, cb)[1], OM.eform_meter(p_drop, cb)[1]
        assert full > dropped * 1.01, (full, dropped)


@pytest.mark.gpu
@pytest.mark.parametrize("scheme,bits,case", PARAMS)
def test_meter_counts_a_huge_bound_on_an_underflowed_weight(scheme, bits, case):
    import paper_2607_28699_gb300 as wc
    c = build_case(scheme, bits, case)
    wl, od = c["wl"], c["od"]
    gd = wc.CacheDesc(num_q_heads=4, num_kv_heads=1, num_pages=wl.num_pages, scheme=scheme, dither_bits=bits,
                      seed=9)
    gcache = numpy_cache_to_gpu(c["cache"], gd)
    ws = wc.Workspace(gd, 1, wl.max_pages)
    ctx = torch.tensor([S], dtype=torch.int32, device="cuda")
    q = torch.from_numpy(c["q16"]).cuda()
    bt = torch.from_numpy(c["bt"]).cuda()
    tier_b = scheme != 1
    if tier_b:
        out, meter, raw, meter_b, raw_b = wc.metered_decode_attention_tier_b(gd, 0, q, bt, ctx, gcache, ws,
                                                                            DELTA_LOC)
    else:
        out, meter, raw = wc.metered_decode_attention(gd, 0, q, bt, ctx, gcache, ws)
    torch.cuda.synchronize()
    assert wc.read_status(ws) == 0
    r = OP.decode_sequence(od, 0, c["q16"][0], c["bt"][0], S, c["cache"], delta_loc=DELTA_LOC if tier_b else None)
    pairs = [("meter_raw", raw, "meter_raw", "meter", meter)]
    if tier_b:
        pairs.append(("meter_b_raw", raw_b, "meter_b_raw", "meter_b", meter_b))
    for what, g_raw, key, mkey, g_meter in pairs:
        g = g_raw.cpu().numpy()[0].astype(np.float64)
        assert not np.any(np.isnan(g)), f"{what}: NaN"
        ref = r[key]
        with np.errstate(over="ignore"):                    # the GPU's fp32: +inf past its range
            ref32 = ref.astype(np.float32).astype(np.float64)
        assert_close(g, ref32, what)
        assert_sound(g, ref, None, what)
        assert_close(g_meter.cpu().numpy()[0], r[mkey], what.replace("_raw", ""))
    assert_close(out.cpu().numpy()[0], r["out"], "out")
