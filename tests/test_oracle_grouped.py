"""Pins for the oracle's grouped-scale cache with the fixed-channel outlier
bypass (§6.2.3 "Storage side" and §6.2.5 "Fixed-channel outlier bypass"): one group
of 128 channels and no bypass is the per-token scheme; each 32-channel group
is the per-token quantizer run on its own channels; bypassed channels are
exact and leave the group amax (no clipping elsewhere); the byte accounts of
Tables "granularity" and "bypassbudget"; the grouped Tier-B proxy against the
measured logit-error variance over dither seeds; the controlled experiment of
Table "amax" (massive pairs need the amax exclusion); the pair calibration;
and the meter's soundness on grouped caches."""

import os

import numpy as np
import pytest

import workloads as W
from oracle import meter as M
from oracle import philox
from oracle import pipeline as OP
from oracle import quantizer as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "storage_bytes.txt")


def _golden(kind):
    out = []
    for line in open(GOLDEN):
        f = line.split()
        if f and f[0] == kind:
            out.append([float(x) for x in f[1:]])
    return out


def _rows(rng, n, d=128):
    scale = np.exp(rng.normal(0.0, 0.5, d))
    return (rng.standard_normal((n, d)) * scale).astype(np.float16)


def _cache(scheme, k, v, slots, m=0, G=32, pairs=None, seed=9, layout=0, exclude=True):
    n, hkv = k.shape[0], k.shape[1]
    od = OP.Desc(num_q_heads=hkv, num_kv_heads=hkv, num_pages=(max(slots) // 16) + 1, scheme=scheme, seed=seed,
                 group_channels=G, num_bypass_pairs=m, rope_layout=layout)
    c = OP.empty_cache(od)
    if not exclude:                       # the "amax unchanged" control of Table "amax"
        orig = Q.group_scales
        Q.group_scales = lambda x, g, e=(), exclude_from_amax=True: orig(x, g, e, False)
        try:
            OP.write_tokens(od, 0, k, v, slots, c, bypass_pairs=pairs)
        finally:
            Q.group_scales = orig
    else:
        OP.write_tokens(od, 0, k, v, slots, c, bypass_pairs=pairs)
    return od, c


def _xi_storage_order(seed, layer, kv_head, slots, tag):
    """The dither by channel of the grouped scheme, built independently: the
    Philox bytes in storage order, moved to the channel each position holds."""
    xi_pos = philox.dither_values(philox.dither_integers(seed, layer, kv_head, slots, tag, 128, 8), 8)
    xi = np.zeros_like(xi_pos)
    for p in range(128):
        if tag == 0:
            c, ks, j = p // 32, (p // 4) % 8, p % 4
            xi[:, 16 * ks + 4 * c + j] = xi_pos[:, p]
        else:
            g, mt, e = p // 16, (p // 2) % 8, p % 2
            xi[:, 16 * mt + 8 * e + g] = xi_pos[:, p]
    return xi


def test_storage_orders_are_permutations_with_whole_groups_per_fragment_step():
    for tag in (0, 1):
        o = OP.storage_order(128, tag)
        assert sorted(o) == list(range(128))
    ok, ov = OP.storage_order(128, 0), OP.storage_order(128, 1)
    for ks in range(8):       # K: positions 32c + 4ks + j (c, j = 0..3) are one QK k-step
        assert len({ok[32 * c + 4 * ks + j] // 32 for c in range(4) for j in range(4)}) == 1
    for mt in range(8):       # V: positions 16g + 2mt + e (g = 0..7, e = 0, 1) are one PV m-tile
        assert {ov[16 * g + 2 * mt + e] for g in range(8) for e in range(2)} == set(range(16 * mt, 16 * mt + 16))


def test_one_group_without_bypass_is_the_per_token_quantizer():
    rng = np.random.default_rng(0)
    k, v = _rows(rng, 40 * 2).reshape(40, 2, 128), _rows(rng, 40 * 2).reshape(40, 2, 128)
    slots = rng.permutation(64)[:40]
    od, b = _cache(OP.SCHEME_DITHER_INT8_G32, k, v, slots, G=128)
    page, off = slots // 16, slots % 16
    for h in range(2):
        for tag, x, name in ((0, k, "k"), (1, v, "v")):
            s = Q.int8_scale(x[:, h])
            xi = _xi_storage_order(od.seed, 0, h, slots, tag)
            code = Q.dither_code(x[:, h], s, xi)
            assert np.array_equal(b[name + "_scale"][page, h, off][:, 0], s)
            assert np.array_equal(b[name + "_codes"][page, h, off], code[:, OP.storage_order(128, tag)])
            if tag == 0:
                r = Q.dither_reconstruct(code, s, xi) - x[:, h].astype(np.float64)
                assert np.array_equal(b["k_witness"][page, h, off], Q.witness(r, 8, 0))


def test_each_group_is_the_per_token_quantizer_on_its_channels():
    rng = np.random.default_rng(1)
    x = _rows(rng, 50)
    x[3] = 0
    x[7, 32:64] = 0                                            # an all-zero group
    slots = np.arange(50) + 100
    desc = OP.Desc(scheme=OP.SCHEME_DITHER_INT8_G32)
    code, s, rec = OP.quantize_rows(desc, 2, 1, x, slots, 0)
    xi = _xi_storage_order(desc.seed, 2, 1, slots, 0)
    for g in range(4):
        sl = slice(32 * g, 32 * g + 32)
        s_ref = Q.int8_scale(x[:, sl])
        assert np.array_equal(s[:, g], s_ref)
        assert np.array_equal(code[:, sl], Q.dither_code(x[:, sl], s_ref, xi[:, sl]))
        assert np.array_equal(rec[:, sl], Q.dither_reconstruct(code[:, sl], s_ref, xi[:, sl]))
    assert np.all(s[7, 1] == 0) and np.all(code[7, 32:64] == 0)


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
def test_bypassed_channels_exact_and_out_of_the_amax(layout):
    rng = np.random.default_rng(2)
    x = _rows(rng, 60)
    pairs = np.array([3, 17, 40, 58])
    dims = Q.bypass_dims(pairs, 128, layout)
    x[:, dims] = (rng.standard_normal((60, 8)) * 300).astype(np.float16)      # massive channels
    desc = OP.Desc(scheme=OP.SCHEME_DITHER_INT8_G32, num_bypass_pairs=4, rope_layout=layout)
    slots = np.arange(60)
    code, s, rec = OP.quantize_rows(desc, 0, 0, x, slots, 0, dims)
    x64 = x.astype(np.float64)
    assert np.array_equal(rec[:, dims], x64[:, dims]) and np.all(code[:, dims] == 0)
    keep = np.setdiff1d(np.arange(128), dims)
    for t in range(60):                                        # amax over the kept channels, brute force
        for g in range(4):
            ch = [c for c in range(32 * g, 32 * g + 32) if c not in set(dims)]
            assert s[t, g] == Q.scale_of_amax(np.max(np.abs(x64[t, ch])))
    s_chan = np.repeat(s, 32, axis=1).astype(np.float64)
    r = rec - x64
    assert np.all(np.abs(r[:, keep]) <= s_chan[:, keep] / 2)  # no clipping (§4.2 "never clips")
    # the witness of the written cache: band norms of the residual, exact channels contributing 0
    k = np.stack([x, x], axis=1)
    od, c = _cache(OP.SCHEME_DITHER_INT8_G32, k, k, slots, m=4, pairs=np.stack([pairs, pairs]), layout=layout,
                   seed=desc.seed)
    rows = lambda name, width: c[name][:, 0].reshape(-1, width)[:60]          # KV head 0, slots 0 .. 59
    assert np.array_equal(rows("k_witness", 8), Q.witness(r, 8, layout))
    assert np.array_equal(rows("k_bypass", 8), x[:, dims])
    # values have no bypass: grouped scales over all their channels
    assert np.array_equal(rows("v_scale", 4), Q.group_scales(x, 32))


def test_byte_accounts_match_the_paper_tables():
    for G, kv_bytes in _golden("granularity"):
        od = OP.Desc(scheme=OP.SCHEME_DITHER_INT8_G32, group_channels=int(G), num_pages=1, num_kv_heads=1)
        c = OP.empty_cache(od)
        per = lambda name: c[name].nbytes // 16                 # bytes per token-head
        assert per("k_codes") + per("k_scale") + per("v_codes") + per("v_scale") == kv_bytes
    for m, kbytes, saved in _golden("bypass"):
        od = OP.Desc(scheme=OP.SCHEME_DITHER_INT8_G32, num_bypass_pairs=int(m), num_pages=1, num_kv_heads=1)
        c = OP.empty_cache(od)
        b = (c["k_codes"].nbytes + c["k_scale"].nbytes + c["k_bypass"].nbytes) // 16
        assert b == kbytes
        assert round(100 * (1 - b / 256), 1) == saved


def test_grouped_proxy_equals_measured_logit_error_variance():
    rng = np.random.default_rng(3)
    k = _rows(rng, 8)
    pairs = np.array([5, 30])
    dims = Q.bypass_dims(pairs, 128, Q.ROPE_HALF)
    k[:, dims] *= 40
    q = rng.standard_normal(128)
    q[dims] *= 10                     # the exact channels must carry no variance, however large q is there
    slots = np.arange(8)
    errs = []
    for seed in range(1500):
        desc = OP.Desc(num_kv_heads=1, num_q_heads=1, seed=seed, scheme=OP.SCHEME_DITHER_INT8_G32,
                       num_bypass_pairs=2)
        _, s, khat = OP.quantize_rows(desc, 3, 0, k, slots, 0, dims)
        errs.append((khat - k.astype(np.float64)) @ q / np.sqrt(128))
    errs = np.array(errs)
    u = M.tier_b_bound_grouped(q, s, 32, dims, ctx_len=8, delta_loc=0.05)
    proxy = u * u / (2 * np.log(2 * 8 / 0.05))
    measured = errs.var(axis=0)
    assert np.all(np.abs(measured / proxy - 1) < 0.15), measured / proxy
    # one group, no bypass: the per-token proxy
    s1 = Q.int8_scale(k)
    assert np.allclose(M.tier_b_bound_grouped(q, s1[:, None], 128, [], 8, 0.05),
                       M.tier_b_bound(q, s1.astype(np.float64), 8, 0.05), rtol=1e-12)


def test_massive_pairs_need_the_amax_exclusion():
    """Table "amax": with 4 injected massive RoPE pairs, bypassing them alone
    barely moves the certificate; bypass plus amax exclusion collapses it."""
    rng = np.random.default_rng(4)
    S, hkv = 512, 2
    pairs = np.array([[3, 10, 20, 25], [1, 12, 22, 30]])
    k = np.stack([_rows(rng, S) for _ in range(hkv)], axis=1).astype(np.float64)
    for h in range(hkv):
        dims = Q.bypass_dims(pairs[h], 128, Q.ROPE_HALF)
        k[:, h, dims] = rng.choice([-1, 1], (S, 8)) * rng.uniform(50, 70, (S, 8))
    k = k.astype(np.float16)
    v = np.stack([_rows(rng, S) for _ in range(hkv)], axis=1)
    slots = np.arange(S)
    qs = rng.standard_normal((16, 2, 128)).astype(np.float16)
    bt = np.arange(S // 16)
    meters = {}
    for name, m, excl in (("none", 0, True), ("bypass_only", 4, False), ("bypass_excluded", 4, True)):
        od, c = _cache(OP.SCHEME_DITHER_INT8_G32, k, v, slots, m=m, pairs=pairs[:, :m] if m else None,
                       exclude=excl)
        mb = []
        for q in qs:
            r = OP.decode_sequence(od, 0, q, bt, S, c, delta_loc=1e-4)
            mb.extend(r["meter_b_raw"])
        meters[name] = np.array(mb)
    med = {n: float(np.median(x)) for n, x in meters.items()}
    cov = {n: float(np.mean(x <= 0.2)) for n, x in meters.items()}
    assert med["none"] > 0.5 and cov["none"] <= 0.1
    assert 0.75 * med["none"] < med["bypass_only"] < med["none"]           # a few percent at most
    assert med["bypass_excluded"] < med["none"] / 10 and cov["bypass_excluded"] >= 0.95


@pytest.mark.parametrize("layout", [Q.ROPE_HALF, Q.ROPE_INTERLEAVED])
def test_calibration_selects_the_massive_pairs(layout):
    rng = np.random.default_rng(5)
    x = _rows(rng, 200).astype(np.float64)
    pairs = np.array([2, 9, 33, 61])
    x[:, Q.bypass_dims(pairs, 128, layout)] *= 30
    assert np.array_equal(Q.select_bypass_pairs(x.astype(np.float16), 4, layout), pairs)
    assert np.array_equal(Q.select_bypass_pairs(x.astype(np.float16), 2, layout),
                          np.sort(pairs[np.argsort(-np.sum(x[:, Q.bypass_dims(pairs, 128, layout)].reshape(200, 4, 2) ** 2,
                                                           axis=(0, 2)))[:2]]))
    assert len(Q.select_bypass_pairs(x.astype(np.float16), 0, layout)) == 0
    # a pair's energy is that of both its dims: here only the second dim is large
    y = rng.standard_normal((200, 128))                       # unit channels: the margins are clear
    second = Q.bypass_dims(pairs, 128, layout).reshape(4, 2)[:, 1]
    y[:, second] *= 30
    y[:, Q.bypass_dims(np.array([5, 6, 7, 8]), 128, layout).reshape(4, 2)[:, 0]] *= 10
    assert np.array_equal(Q.select_bypass_pairs(y.astype(np.float16), 4, layout), pairs)


@pytest.mark.parametrize("m", [0, 4])
def test_meter_sound_on_grouped_caches(m):
    wl = W.Workload("g", 1, 8, 2, [300, 77], shuffle_pages=True, seed=6)
    bt = W.block_tables(wl)
    sm = W.slot_mapping(wl, bt)
    k, v = W.layer_kv(wl, 0)
    k = k.numpy().copy()
    pairs = np.array([[4, 11, 40, 60], [0, 7, 19, 33]])[:, :m]
    if m:
        for h in range(2):
            k[:, h, Q.bypass_dims(pairs[h], 128, Q.ROPE_HALF)] *= 20
    q = W.layer_queries(wl, 0).numpy()
    od = OP.Desc(num_q_heads=8, num_kv_heads=2, num_pages=wl.num_pages, scheme=OP.SCHEME_DITHER_INT8_G32, seed=9,
                 num_bypass_pairs=m)
    cache = OP.empty_cache(od)
    OP.write_tokens(od, 0, k, v.numpy(), sm, cache, bypass_pairs=pairs if m else None)
    offs = np.concatenate([[0], np.cumsum(wl.ctx_lens)[:-1]])
    for b, S in enumerate(wl.ctx_lens):
        for scale in (1.0, 4.0):
            r = OP.decode_sequence(od, 0, q[b] * scale, bt[b], S, cache, k[offs[b]:offs[b] + S],
                                   v.numpy()[offs[b]:offs[b] + S])
            assert np.all(r["tv"] <= r["meter_raw"] * (1 + 1e-12))


def test_storage_round_trip():
    """reconstruct() of a written grouped cache gives back the quantizer's
    channel-order reconstruction exactly (keys with the bypass, values)."""
    rng = np.random.default_rng(7)
    n = 37
    k = np.stack([_rows(rng, n), _rows(rng, n)], axis=1)
    v = np.stack([_rows(rng, n), _rows(rng, n)], axis=1)
    slots = rng.permutation(80)[:n]
    pairs = np.array([[1, 2, 30, 63], [4, 5, 6, 7]])
    od, c = _cache(OP.SCHEME_DITHER_INT8_G32, k, v, slots, m=4, pairs=pairs)
    for h in range(2):
        dims = Q.bypass_dims(pairs[h], 128, Q.ROPE_HALF)
        _, _, krec = OP.quantize_rows(od, 0, h, k[:, h], slots, 0, dims)
        _, _, vrec = OP.quantize_rows(od, 0, h, v[:, h], slots, 1)
        khat, vhat, _ = OP.reconstruct(od, 0, h, slots, c)
        assert np.array_equal(khat, krec) and np.array_equal(vhat, vrec)
