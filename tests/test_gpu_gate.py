"""GPU gate (wc_gate) equals the oracle's gate bit for bit on the same fp32
meter_raw input, including ties at tau, +inf and NaN."""

import numpy as np
import pytest
import torch

from oracle import meter as M

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("group,n", [(7, 28 * 28 * 32), (4, 8), (1, 1), (7, 0)])
def test_gate_bit_exact(group, n):
    import paper_2607_28699_gb300 as wc
    rng = np.random.default_rng(group * 1000 + n)
    mr = np.exp(rng.normal(-2.5, 1.5, n)).astype(np.float32)
    if n >= 8:
        mr[::13] = np.float32(0.1)                      # ties at tau keep
        mr[1::17] = np.inf
        mr[2::19] = np.nan
    for tau in (0.05, 0.1, 0.2, 1.0, 5.0):
        keep_q, keep_kv, kept = wc.gate(torch.from_numpy(mr).cuda(), group, tau)
        oq, okv, nq, nkv = M.gate(mr, tau, group)
        assert np.array_equal(keep_q.cpu().numpy().astype(bool), oq)
        assert np.array_equal(keep_kv.cpu().numpy().astype(bool), okv)
        assert kept.cpu().tolist() == [nq, nkv]
