"""Plain fp64 CPU oracle for the WitCert hot path (arxiv 2607.28699).

TEST INFRASTRUCTURE ONLY.  Nothing in the product package may import,
call or execute this package; only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.
It shares no code with the CUDA path: every step below is written from the
paper's definitions, in numpy float64 (or exact integer / rational
arithmetic where the definition is a rounding rule), without blocking,
fusion or reordering beyond what the definitions state.

Modules
-------
fp         fp16 round-to-nearest / round-up, OCP fp8-e4m3fn encode/decode.
philox     Philox4x32-10 (Salmon et al., SC'11) and the dither derived from it
           (§6.2.1 "Research kernels": Philox dither from a slot-keyed counter;
           §6.2.3 storage side: counter uses the slot, not the position).
quantizer  subtractive-dither INT8 quantizer (§4.2 "Subtractive dither"),
           raw-cast fp8, residual band-norm witness (§4.1 Eq. witness),
           value witness (§3 output bound), grouped scales with the
           fixed-channel outlier-pair bypass and its calibration (§6.2.3).
meter      exact / compressed attention, total variation (§3 setup), the
           flawed dispersion certificate (§3 Eq. flawed, regression guard),
           Tier-A logit bound (§4.1 Thm. "Sound black-box logit bound"),
           Tier-B sub-Gaussian bound, per-token and grouped (§4.2), the
           e-form meter (§3 Thm. "Sound replacement"), the value term,
           output bound and joint gate (§3, §4.2), block-level repair
           selection (§6.3.5), gate (§6 meter loop box).
pipeline   the write path over a paged cache (per-token, fp8 and grouped
           schemes) and the metered decode step, composed from the
           functions above.

Every function is pinned by ``tests/test_oracle_*.py`` against something
other than itself (paper-printed values, library routines, exact rational
arithmetic, closed forms, invariants, brute force).
"""

from . import fp, philox, quantizer, meter, pipeline  # noqa: F401,E402
