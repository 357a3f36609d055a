"""Attention, total variation, the Tier-A bound, the e-form meter and the gate.

Test infrastructure only (see ``oracle/__init__.py``).  All arithmetic is
float64 and follows the definitions in the order the paper states them.

§3 setup: p and p~ are the softmax distributions over the cached tokens
computed from exact and compressed keys; eps_t is token t's logit error;
c_t >= |eps_t| is any per-token bound; TV(p, p~) = 1/2 sum_t |p_t - p~_t|.
The machine-checked statement (Appendix A, "L1 main theorem") fixes the
sign convention p_t = p~_t exp(-eps_t) / Z, i.e. eps_t = z~_t - z_t.

§3 Thm. "Sound replacement": A = E_p~[e^c] and TV <= 1/2 (A^2 - 1).
The meter is reported as min(1, .) (§4.3) and evaluated without truncating
c; +inf on overflow is sound and counts as over threshold (§6.2.5, on
fp32 overflow).  Here 1/2 (A^2 - 1) is computed as 1/2 D (D + 2) with
D = A - 1 = E_p~[expm1(c)], which is the same number without the
cancellation of A^2 - 1 for small c (reading: the paper only asks for a
numerically careful evaluation, "in the log domain").  From logits
(eform_terms, the pipeline's form) a term p~_t expm1(c_t) that float64
cannot form as a product (p~_t underflowing, expm1(c_t) overflowing) is taken
in the log domain, so it keeps its value instead of 0 or +inf.

§4.1 Thm. "Sound black-box logit bound": |eps_t| = |q . r_t| / sqrt(d)
<= (1/sqrt(d)) sum_b ||q_b|| w_{t,b} =: c_t.

§4.2 Tier B (controlled quantizer, subtractive dither): Lemma "Uniform
sub-Gaussian proxy" gives the logit error of token t the variance proxy
varsigma_t^2 = (1/d) sum_c q_c^2 s_{c,t}^2 / 12, and with probability at
least 1 - delta_loc jointly over the S tokens |eps_t| <= u_t =
sqrt(2 varsigma_t^2 log(2S / delta_loc)); u_t then replaces c_t in the
e-form meter.  Here the scale is one stored fp16 value per (token, KV head)
(§6.2.2 per-token granularity), so varsigma_t^2 = ||q||^2 s_t^2 / (12 d).
The guarantee is probabilistic and holds for non-adaptive queries (§4.2
"Scope of the probabilistic guarantee").  With grouped scales (§6.2.3) the
scale of channel c is its group's, and a bypassed channel is exact, so it
carries no error: varsigma_t^2 = (1/(12 d)) sum_{c not bypassed} q_c^2 s_{g(c),t}^2.

§3 output propagation and §4.2 "Value side and the joint event": with
rho^v_t = ||v^_t - v_t||, ||y - y^|| <= 2 TV max_t ||v_t|| + sum_t p~_t rho^v_t;
with TV bounded by the meter this is an output-error bound computable from
stored per-token values.  Reading (the paper names pass_V without a
formula): pass_V holds when the value term sum_t p~_t rho^v_t is at most
tau_V max_t ||v_t||, and the joint gate keeps a cell iff pass_K (meter_raw
<= tau_K) and pass_V, both decided in float32.

§6.3.5 "Block-level paging": the e-form certificate is block decomposable.
With p~ held fixed, replacing page j's keys by their exact values sets c_t = 0
for its tokens and lowers D = A - 1 by exactly C_j = sum_{t in j} p~_t
expm1(c_t).  Paging in pages by decreasing C_j until 1/2 D (D + 2) <= tau
uses the fewest pages (all C_j >= 0).  Reading: ties in C_j go to the lower
logical page index.

Gate (§6 meter-loop box; §4.3 certified vs risk-ranked): a (layer, head)
falls back when its meter exceeds tau.  Reading: keep the compressed path
iff meter_raw <= tau (so equality keeps, NaN falls back), evaluated in
float32 on the float32 meter_raw; a KV head keeps its compressed cache only
if all G query heads sharing it keep (any-of-G fallback, §5 statistics "at
KV-head any-of-G granularity").
"""

import numpy as np

from . import quantizer


def softmax(z):
    z = np.asarray(z, dtype=np.float64)
    m = np.max(z, axis=-1, keepdims=True)
    e = np.exp(z - m)
    return e / np.sum(e, axis=-1, keepdims=True)


def total_variation(p, p_tilde):
    return 0.5 * np.sum(np.abs(np.asarray(p) - np.asarray(p_tilde)), axis=-1)


def perturbed(p_tilde, eps):
    """p_t = p~_t exp(-eps_t) / Z (Appendix A, L1 hypothesis)."""
    w = np.asarray(p_tilde, dtype=np.float64) * np.exp(-np.asarray(eps, dtype=np.float64))
    return w / np.sum(w, axis=-1, keepdims=True)


def flawed_bound(p_tilde, c):
    """§3 Eq. (flawed): 1/2 e^{2 cmax} (E|c - cbar| + cbar (e^{cmax} - 1)).

    Unsound; kept only so the tests can show the paper's counterexample.
    """
    p_tilde = np.asarray(p_tilde, dtype=np.float64)
    c = np.asarray(c, dtype=np.float64)
    cbar = np.sum(p_tilde * c, axis=-1)
    cmax = np.max(c, axis=-1)
    disp = np.sum(p_tilde * np.abs(c - cbar[..., None]), axis=-1)
    return 0.5 * np.exp(2 * cmax) * (disp + cbar * np.expm1(cmax))


def eform_meter(p_tilde, c):
    """Returns (meter, meter_raw, A) for A = E_p~[e^c]."""
    p_tilde = np.asarray(p_tilde, dtype=np.float64)
    c = np.asarray(c, dtype=np.float64)
    with np.errstate(over="ignore", invalid="ignore"):
        terms = p_tilde * np.expm1(c)
        terms = np.where(p_tilde == 0, 0.0, terms)      # 0 * e^huge is 0 mass
    return meter_of_terms(terms)


def meter_of_terms(terms):
    """(meter, meter_raw, A) from the terms p~_t expm1(c_t) of D = A - 1."""
    with np.errstate(over="ignore", invalid="ignore"):
        D = np.sum(terms, axis=-1)
        raw = 0.5 * D * (D + 2.0)
    raw = np.where(np.isnan(raw), np.inf, raw)
    return np.minimum(1.0, raw), raw, 1.0 + D


def eform_terms(z, c):
    """p~ = softmax(z) and the terms p~_t expm1(c_t) of D, for logits z of
    cached tokens (all finite) and bounds c >= 0.

    The product p~_t expm1(c_t) is the definition as written; where float64
    cannot hold it (p~_t underflows to 0 for a logit ~745 below the maximum,
    or expm1(c_t) overflows for c_t > ~709) the same number is taken in the
    log domain, exp(log p~_t + log expm1(c_t)) with log p~_t = z_t - m -
    log sum_s e^{z_s - m} and log expm1(c) = c + log(-expm1(-c)), so a token
    whose weight underflows still counts with its bound.  Elsewhere the terms
    are bit for bit those of eform_meter(softmax(z), c).
    """
    z = np.asarray(z, np.float64)
    c = np.asarray(c, np.float64)
    p = softmax(z)
    m = np.max(z, axis=-1, keepdims=True)
    with np.errstate(over="ignore", invalid="ignore", divide="ignore"):
        em1 = np.expm1(c)
        direct = p * em1
        log_p = (z - m) - np.log(np.sum(np.exp(z - m), axis=-1, keepdims=True))
        logged = np.exp(log_p + c + np.log(-np.expm1(-c)))
        terms = np.where((p > 0) & np.isfinite(em1), direct, logged)
    return p, terms


def eform_meter_logits(z, c):
    """eform_meter of softmax(z) with the terms of eform_terms: (meter, meter_raw, A)."""
    return meter_of_terms(eform_terms(z, c)[1])


def tier_a_bound(q, w, num_bands, rope_layout):
    """c_t = (1/sqrt(d)) sum_b ||q_b|| w_{t,b}.

    q: [..., d]; w: [..., S, B] stored witness; returns [..., S].
    """
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    qn = quantizer.band_norms(q, num_bands, rope_layout)          # [..., B]
    w = np.asarray(w, dtype=np.float64)
    return np.einsum("...b,...sb->...s", qn, w) / np.sqrt(d)


def tier_b_bound(q, s, ctx_len, delta_loc):
    """u_t = sqrt(2 varsigma_t^2 log(2 S / delta_loc)), varsigma_t^2 = ||q||^2 s_t^2 / (12 d).

    q: [..., d] query; s: [..., S] stored K scales of the S tokens; returns [..., S].
    """
    q = np.asarray(q, dtype=np.float64)
    d = q.shape[-1]
    s = np.asarray(s, dtype=np.float64)
    var = np.sum(q * q, axis=-1)[..., None] * s * s / (12.0 * d)
    return np.sqrt(2.0 * var * np.log(2.0 * ctx_len / delta_loc))


def tier_b_bound_grouped(q, s_groups, group, excluded, ctx_len, delta_loc):
    """u_t with grouped scales and bypassed channels (exact, no error).

    q: [d]; s_groups: [S, d / group] stored fp16 group scales; excluded: the
    bypassed dims; returns [S].
    """
    q = np.asarray(q, dtype=np.float64).copy()
    d = q.shape[-1]
    q[np.asarray(excluded, dtype=np.int64)] = 0.0
    qn2 = np.sum((q * q).reshape(d // group, group), axis=-1)            # [G]
    sg = np.asarray(s_groups, dtype=np.float64)
    var = (sg * sg) @ qn2 / (12.0 * d)
    return np.sqrt(2.0 * var * np.log(2.0 * ctx_len / delta_loc))


def value_term(p_tilde, rho):
    """sum_t p~_t rho^v_t."""
    return np.sum(np.asarray(p_tilde, np.float64) * np.asarray(rho, np.float64), axis=-1)


def output_bound(meter, v_max, vterm):
    """||y - y^|| <= 2 TV max_t ||v_t|| + sum_t p~_t rho^v_t, with TV <= meter (<= 1)."""
    return 2.0 * np.asarray(meter, np.float64) * np.asarray(v_max, np.float64) + np.asarray(vterm, np.float64)


def logits(q, k):
    """z_t = q . k_t / sqrt(d); q [..., d], k [..., S, d] -> [..., S]."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    return np.einsum("...d,...sd->...s", q, k) / np.sqrt(q.shape[-1])


def attend(p, v):
    """y = sum_t p_t v_t."""
    return np.einsum("...s,...sd->...d", np.asarray(p, np.float64), np.asarray(v, np.float64))


def gate(meter_raw, tau, group):
    """Keep/fallback decisions from float32 meter_raw [..., n_cells].

    Returns keep_q (bool, per query-head cell), keep_kv (bool, per group of
    ``group`` consecutive cells) and the two kept counts.
    """
    mr = np.asarray(meter_raw, dtype=np.float32)
    keep_q = mr <= np.float32(tau)
    n = keep_q.shape[-1]
    if n % group:
        raise ValueError("cells must come in whole groups")
    keep_kv = np.all(keep_q.reshape(keep_q.shape[:-1] + (n // group, group)), axis=-1)
    return keep_q, keep_kv, int(np.sum(keep_q)), int(np.sum(keep_kv))


def joint_gate(meter_raw, vterm, v_max, tau_k, tau_v, group):
    """Joint keep decisions (pass_K and pass_V) in float32, with the same
    layout and counts as ``gate``."""
    mr = np.asarray(meter_raw, dtype=np.float32)
    vt = np.asarray(vterm, dtype=np.float32)
    vm = np.asarray(v_max, dtype=np.float32)
    keep_q = (mr <= np.float32(tau_k)) & (vt <= np.float32(tau_v) * vm)
    n = keep_q.shape[-1]
    if n % group:
        raise ValueError("cells must come in whole groups")
    keep_kv = np.all(keep_q.reshape(keep_q.shape[:-1] + (n // group, group)), axis=-1)
    return keep_q, keep_kv, int(np.sum(keep_q)), int(np.sum(keep_kv))


def page_contributions(p_tilde, c, page_of_token, n_pages, terms=None):
    """C_j = sum over the tokens of logical page j of p~_t expm1(c_t) (the
    terms may be given, e.g. those of eform_terms)."""
    if terms is None:
        p_tilde = np.asarray(p_tilde, np.float64)
        with np.errstate(over="ignore", invalid="ignore"):
            terms = p_tilde * np.expm1(np.asarray(c, np.float64))
            terms = np.where(p_tilde == 0, 0.0, terms)      # as in eform_meter
    return np.bincount(np.asarray(page_of_token, dtype=np.int64), weights=terms, minlength=n_pages)


def repair_plan(contrib, tau):
    """Fewest pages whose exact values bring the meter to tau or below.

    Pages rank by decreasing C_j (NaN first, ties to the lower index); the
    remaining excess after paging in the first k is R_k = the sum of the
    contributions not yet paged in, and k is the least with
    1/2 R_k (R_k + 2) <= tau (all pages when tau < 0).
    Returns (pages in paging order, R_k).
    """
    C = np.asarray(contrib, np.float64)
    n = len(C)
    order = sorted(range(n), key=lambda j: (not np.isnan(C[j]), 0.0 if np.isnan(C[j]) else -C[j], j))
    sorted_c = C[order]
    # R[k] = sum(sorted_c[k:]), R[n] = 0
    R = np.concatenate([np.cumsum(sorted_c[::-1])[::-1], [0.0]])
    with np.errstate(invalid="ignore", over="ignore"):
        ok = 0.5 * R * (R + 2.0) <= tau
    k = int(np.argmax(ok)) if np.any(ok) else n
    return [int(j) for j in order[:k]], float(R[k])
