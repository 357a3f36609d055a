"""Write-path quantizers and the band-norm residual witness.

Test infrastructure only (see ``oracle/__init__.py``).

Subtractive-dither INT8 (§4.2 "Subtractive dither"; §6.2.1 research write
kernel; per-token scalar scale of the SGLang integration, §6.2.2):

  amax = max_c |x_c|                       over one token's head_dim values
  s    = fp16_rn( fp32(amax) / 126.5f )    Q - 1/2 with Q = 127; the stored
                                           fp16 scale is the one quantized
                                           with (§6.2.1: quantizing with an
                                           fp32 scale while storing fp16
                                           breaks |err| <= s/2)
  code = round_half_even( x/s + xi )       exact real arithmetic, then
                                           clamped to [-127, 127]
  x^   = s * (code - xi)

Readings where the paper is silent: ties of the exact value x/s + xi go to
the even integer; s that rounds to 0 while amax > 0 is raised to the least
fp16 subnormal 2^-24 (then clipping can occur, and the witness, being the
actual residual, stays sound); amax = 0 gives s = 0, code 0, x^ = 0.

Grouped scales with a fixed-channel outlier bypass (§6.2.3 "Storage side",
Table "granularity"; §6.2.5 "Fixed-channel outlier bypass", Tables "amax" and
"bypassbudget"): one fp16 scale per token and group of G_c contiguous
channels (G_c = 32 by default), s_g = fp16_rn(fp32(amax_g) / 126.5f) by the
rule above, where amax_g leaves out the bypassed channels; the bypassed
channels are the 2m dims of m RoPE pairs fixed per (layer, KV head), stored
exactly as fp16 (x^ = x there) with code 0.  Readings: the bypass is a key
side device (RoPE pairs), values use the grouped scales only; a group whose
channels are all bypassed gets s = 0.

Raw-cast fp8-e4m3 (the black-box fp8 scheme of Fig. f5): code = e4m3(x),
x^ = decode(code), no scale, no dither.

Witness (§4.1, Eq. witness, Lemma "RoPE band unitarity"): r = x^ - x,
w_b = ||r_b|| over the coordinates of band b, stored in fp16 rounded up.
The d/2 RoPE frequency pairs are grouped into B contiguous bands of
d/(2B) pairs.  Pair j occupies dims (j, j + d/2) in the half-rotation
layout (ROPE_HALF) and dims (2j, 2j+1) in the interleaved layout.
"""

from fractions import Fraction

import numpy as np

from . import fp

ROPE_HALF = 0
ROPE_INTERLEAVED = 1
QMAX = 127
SCALE_DIVISOR = np.float32(126.5)


def int8_scale(x16):
    """Per-row fp16 scale from fp16 rows x16 [..., d] (returns float16 [...])."""
    x = np.asarray(x16, dtype=np.float16).astype(np.float64)
    return scale_of_amax(np.max(np.abs(x), axis=-1))


def scale_of_amax(amax):
    """fp16_rn(fp32(amax) / 126.5f), raised to 2^-24 when it rounds to 0."""
    amax = np.asarray(amax, dtype=np.float64)
    s = (amax.astype(np.float32) / SCALE_DIVISOR).astype(np.float16)
    raise_to_min = (s == 0) & (amax > 0)
    s = np.where(raise_to_min, np.float16(fp.FP16_MIN_SUBNORMAL), s)
    return s.astype(np.float16)


def dither_code(x16, s16, xi):
    """Exact round-half-even of x/s + xi, clamped to [-127, 127].

    x16: fp16 [..., d]; s16: fp16 [...] (one scale per row) or [..., d] (one per
    channel); xi: float64 [..., d] on the grid
    (odd integer) / 2^(bits+1).  All products below are exact in float64:
    s has 11 significant bits and k + 1/2 - xi has at most 20 for |k| <= 255.
    """
    x = np.asarray(x16, dtype=np.float16).astype(np.float64)
    s = np.asarray(s16, dtype=np.float16).astype(np.float64)
    if s.ndim < x.ndim:
        s = s[..., None]
    xi = np.asarray(xi, dtype=np.float64)
    s_b = np.broadcast_to(s, x.shape)
    zero = s_b == 0
    safe_s = np.where(zero, 1.0, s_b)
    est = x / safe_s + xi                      # estimate only
    big = np.abs(est) > 200.0                  # certainly beyond +-127
    k = np.floor(np.clip(est, -200.0, 200.0))
    # make k = floor(x/s + xi) exactly: x >= s*(k - xi) and x < s*(k + 1 - xi)
    for _ in range(2):
        k = np.where(x < safe_s * (k - xi), k - 1, k)
        k = np.where(x >= safe_s * (k + 1 - xi), k + 1, k)
    mid = safe_s * (k + 0.5 - xi)              # exact
    up = x > mid
    tie = x == mid
    odd = np.mod(k, 2) != 0
    code = np.where(up | (tie & odd), k + 1, k)
    code = np.where(big, np.sign(est) * QMAX, code)
    code = np.clip(code, -QMAX, QMAX)
    code = np.where(zero, 0, code)
    return code.astype(np.int8)


def dither_code_fraction(x, s, xi):
    """Scalar exact reference: Python's round() on a Fraction is half-even."""
    if s == 0:
        return 0
    y = Fraction(float(x)) / Fraction(float(s)) + Fraction(float(xi))
    return max(-QMAX, min(QMAX, round(y)))


def dither_reconstruct(code, s16, xi):
    """x^ = s (code - xi), exact in float64 (s per row, or per channel)."""
    s = np.asarray(s16, dtype=np.float16).astype(np.float64)
    if s.ndim < np.ndim(code):
        s = s[..., None]
    return s * (np.asarray(code, dtype=np.float64) - np.asarray(xi, dtype=np.float64))


def bypass_dims(pairs, head_dim, rope_layout):
    """Dims of the bypassed RoPE pairs, pair by pair: [a_0, b_0, a_1, b_1, ...]."""
    pairs = np.asarray(pairs, dtype=np.int64).reshape(-1)
    half = head_dim // 2
    if rope_layout == ROPE_HALF:
        a, b = pairs, pairs + half
    elif rope_layout == ROPE_INTERLEAVED:
        a, b = 2 * pairs, 2 * pairs + 1
    else:
        raise ValueError("unknown rope layout")
    return np.stack([a, b], axis=1).reshape(-1)


def group_scales(x16, group, excluded=(), exclude_from_amax=True):
    """fp16 scale per row and channel group [..., d / group]; the excluded
    (bypassed) channels leave the group amax unless exclude_from_amax is False
    (the "amax unchanged" control of Table "amax")."""
    x = np.abs(np.asarray(x16, dtype=np.float16).astype(np.float64))
    if exclude_from_amax and len(excluded):
        x = x.copy()
        x[..., np.asarray(excluded, dtype=np.int64)] = 0.0
    d = x.shape[-1]
    return scale_of_amax(np.max(x.reshape(x.shape[:-1] + (d // group, group)), axis=-1))


def select_bypass_pairs(k16, m, rope_layout):
    """The m RoPE pairs of largest energy sum_t (x_a^2 + x_b^2) over the rows
    k16 [n, d] (ties to the lower pair), in increasing pair order."""
    x = np.asarray(k16, dtype=np.float16).astype(np.float64)
    d = x.shape[-1]
    pairs = np.arange(d // 2)
    dims = bypass_dims(pairs, d, rope_layout).reshape(-1, 2)
    energy = np.sum(x[:, dims[:, 0]] ** 2 + x[:, dims[:, 1]] ** 2, axis=0)
    order = sorted(pairs, key=lambda j: (-energy[j], j))
    return np.sort(np.asarray(order[:m], dtype=np.int64))


def fp8_quantize(x16):
    """Raw cast to fp8 e4m3fn; returns (codes uint8, x^ float64)."""
    x = np.asarray(x16, dtype=np.float16).astype(np.float64)
    code = fp.e4m3_encode(x)
    return code, fp.e4m3_decode(code)


def band_dims(head_dim, num_bands, rope_layout):
    """Index array [num_bands, dims_per_band] of the dims in each band."""
    pairs = head_dim // 2
    ppb = pairs // num_bands
    out = []
    for b in range(num_bands):
        js = np.arange(b * ppb, (b + 1) * ppb)
        if rope_layout == ROPE_HALF:
            dims = np.concatenate([js, js + pairs])
        elif rope_layout == ROPE_INTERLEAVED:
            dims = np.stack([2 * js, 2 * js + 1], axis=1).reshape(-1)
        else:
            raise ValueError("unknown rope layout")
        out.append(np.sort(dims))
    return np.stack(out)


def band_norms(v, num_bands, rope_layout):
    """Exact-ish float64 per-band Euclidean norms of v [..., d]."""
    v = np.asarray(v, dtype=np.float64)
    dims = band_dims(v.shape[-1], num_bands, rope_layout)
    return np.sqrt(np.sum(v[..., dims] ** 2, axis=-1))


def witness(residual, num_bands, rope_layout):
    """Stored witness: fp16 round-up of the per-band residual norms."""
    return fp.fp16_ru(band_norms(residual, num_bands, rope_layout))


def value_witness(residual, v):
    """Value-side witness of each row (§3 output bound, rho^v_t := ||v^_t - v_t||):
    [..., 2] fp16 = (rho^v rounded up, ||v|| rounded up).  Reading: the value
    norm is stored too (rounded up), so that max_t ||v_t|| in the output bound
    is available at decode time without the exact values."""
    r = np.asarray(residual, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    return np.stack([fp.fp16_ru(np.sqrt(np.sum(r * r, axis=-1))),
                     fp.fp16_ru(np.sqrt(np.sum(v * v, axis=-1)))], axis=-1)
