"""Seeded synthetic inputs shaped like the paper's 7B-class decode workloads.

This module is the only code shared by the CUDA path's tests/benchmark and
the oracle.  It draws inputs and builds page tables; it contains none of the
method's arithmetic (no quantizer, dither, witness, attention or meter).

Recipe (the paper's activations and datasets are not available; these
stand in for Qwen2.5-7B-shaped caches, 28 layers / 28 query / 4 KV heads,
head_dim 128, contexts 4k-128k, §5-§6):

* pre-RoPE K and V rows ~ N(0, 1) * sigma_c with one log-normal(0, 0.5)
  scale per (layer, KV head, channel), drawn separately for K and V, so a
  few channels carry large magnitudes (outlier channels);
* the first token of every sequence (position 0) is an attention sink with
  8x the norm of the others (K and V multiplied by 8 before RoPE);
* K is rotated by RoPE (theta = 1e4, half-rotation pairs (j, j + d/2),
  frequency theta^(-2j/d)) at its position; the cache stores post-RoPE keys;
* the decode query of a sequence of length S is N(0, 1) per dim, rotated at
  position S - 1; in the batch-32 fp8 workload a seeded 5% of
  (sequence, layer, query head) cells get a 4x query;
* tokens of sequence b at positions t occupy slot
  block_table[b, t // 16] * 16 + t % 16; serving workloads shuffle the
  physical page order with a seeded permutation.

Random draws use torch generators so that multi-GB caches can be drawn on
the GPU; draws on the CPU and on a GPU differ, so any comparison draws once
and copies.
"""

from dataclasses import dataclass, field
from typing import List

import numpy as np
import torch

PAGE = 16
HEAD_DIM = 128
ROPE_THETA = 1e4
SCHEME_DITHER_INT8 = 0
SCHEME_FP8_E4M3 = 1


@dataclass
class Workload:
    name: str
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    ctx_lens: List[int]
    scheme: int = SCHEME_DITHER_INT8
    shuffle_pages: bool = False
    taus: List[float] = field(default_factory=lambda: [0.1])
    q_boost_frac: float = 0.0
    seed: int = 0
    head_dim: int = HEAD_DIM
    num_bands: int = 8
    page_size: int = PAGE
    includes_prefill_write: bool = False

    @property
    def batch(self):
        return len(self.ctx_lens)

    @property
    def group(self):
        return self.n_q_heads // self.n_kv_heads

    @property
    def max_pages(self):
        return max((c + self.page_size - 1) // self.page_size for c in self.ctx_lens)

    @property
    def pages_per_seq(self):
        return [(c + self.page_size - 1) // self.page_size for c in self.ctx_lens]

    @property
    def num_pages(self):
        return sum(self.pages_per_seq)

    @property
    def kv_tokens(self):
        """Context tokens read per decode step summed over sequences and layers."""
        return sum(self.ctx_lens) * self.n_layers


def _rng(seed, *salt):
    return np.random.default_rng([seed, *salt])


def config(i, seed=0, ctx_scale=1.0, layers=None):
    """Workload i in 1..5.  ``ctx_scale`` < 1 shrinks contexts for tests
    (results stay ragged: lengths are not rounded to pages)."""
    def ctx(n):
        return max(1, int(round(n * ctx_scale)))

    if i == 1:
        wl = Workload("1L-8q2kv-S4096-dither-int8", 1, 8, 2, [ctx(4096)], seed=seed)
    elif i == 2:
        wl = Workload("28L-28q4kv-S32768-dither-int8-tau0.1", 28, 28, 4, [ctx(32768)], seed=seed)
    elif i == 3:
        r = _rng(seed, 3)
        lens = [ctx(int(x)) for x in r.integers(4096, 8193, size=16)]
        wl = Workload("28L-28q4kv-b16-S4k-8k-paged-shuffled-prefill+decode", 28, 28, 4, lens,
                      shuffle_pages=True, seed=seed, includes_prefill_write=True)
    elif i == 4:
        wl = Workload("28L-28q4kv-S131072-dither-int8", 28, 28, 4, [ctx(131072)], seed=seed)
    elif i == 5:
        r = _rng(seed, 5)
        lens = [ctx(int(x)) for x in r.integers(4096, 32769, size=32)]
        wl = Workload("28L-28q4kv-b32-S4k-32k-fp8-e4m3-witness", 28, 28, 4, lens,
                      scheme=SCHEME_FP8_E4M3, shuffle_pages=True, taus=[0.05, 0.1, 0.2],
                      q_boost_frac=0.05, seed=seed)
    else:
        raise ValueError("configs are numbered 1..5")
    if layers is not None:
        wl.n_layers = layers
    return wl


def block_tables(wl):
    """int32 [batch, max_pages] physical page of each logical page (-1 pad)."""
    order = np.arange(wl.num_pages)
    if wl.shuffle_pages:
        order = _rng(wl.seed, 7).permutation(wl.num_pages)
    bt = np.full((wl.batch, wl.max_pages), -1, dtype=np.int32)
    pos = 0
    for b, n in enumerate(wl.pages_per_seq):
        bt[b, :n] = order[pos:pos + n]
        pos += n
    return bt


def slot_mapping(wl, bt=None):
    """int32 [sum ctx] slots of every token, sequences concatenated."""
    bt = block_tables(wl) if bt is None else bt
    out = []
    for b, S in enumerate(wl.ctx_lens):
        t = np.arange(S)
        out.append(bt[b, t // wl.page_size].astype(np.int64) * wl.page_size + t % wl.page_size)
    return np.concatenate(out).astype(np.int32)


def positions(wl):
    return np.concatenate([np.arange(S) for S in wl.ctx_lens])


def _gen(wl, layer, kind, device):
    g = torch.Generator(device=device)
    g.manual_seed((wl.seed * 1_000_003 + layer * 7919 + kind) % (2 ** 63))
    return g


def rope(x, pos, theta=ROPE_THETA):
    """Rotate x [..., n, d] (float32) by RoPE at integer positions pos [n]."""
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-torch.arange(half, dtype=torch.float64, device=x.device) * 2.0 / d)
    ang = pos.to(torch.float64)[:, None] * inv[None, :]
    cos, sin = torch.cos(ang).to(x.dtype), torch.sin(ang).to(x.dtype)
    while cos.dim() < x.dim():
        cos, sin = cos.unsqueeze(-2), sin.unsqueeze(-2)
    a, b = x[..., :half], x[..., half:]
    return torch.cat([a * cos - b * sin, a * sin + b * cos], dim=-1)


def layer_kv(wl, layer, device="cpu", seq_range=None):
    """Post-RoPE K and V for every token of ``layer``: fp16 [n_tok, Hkv, d].

    ``seq_range`` (lo, hi) restricts to sequences lo..hi-1 (tokens
    concatenated in sequence order).  Draws are made per sequence so a
    restricted draw equals the corresponding slice of the full draw.
    """
    lo, hi = (0, wl.batch) if seq_range is None else seq_range
    H, d = wl.n_kv_heads, wl.head_dim
    gs = _gen(wl, layer, 1, device)
    sig_k = torch.exp(0.5 * torch.randn(H, d, generator=gs, device=device))
    sig_v = torch.exp(0.5 * torch.randn(H, d, generator=gs, device=device))
    ks, vs = [], []
    for b in range(lo, hi):
        S = wl.ctx_lens[b]
        g = _gen(wl, layer, 1000 + b, device)
        k = torch.randn(S, H, d, generator=g, device=device) * sig_k
        v = torch.randn(S, H, d, generator=g, device=device) * sig_v
        if S > 0:   # the sink token (an empty sequence has none)
            k[0] *= 8.0
            v[0] *= 8.0
        pos = torch.arange(S, device=device)
        ks.append(rope(k, pos).to(torch.float16))
        vs.append(v.to(torch.float16))
    return torch.cat(ks), torch.cat(vs)


def layer_queries(wl, layer, device="cpu"):
    """Post-RoPE decode queries fp16 [batch, Hq, d] at positions S - 1."""
    g = _gen(wl, layer, 2, device)
    q = torch.randn(wl.batch, wl.n_q_heads, wl.head_dim, generator=g, device=device)
    if wl.q_boost_frac > 0:
        boost = _rng(wl.seed, 11, layer).random((wl.batch, wl.n_q_heads)) < wl.q_boost_frac
        q = q * torch.where(torch.as_tensor(boost, device=device), 4.0, 1.0)[..., None]
    pos = torch.as_tensor([S - 1 for S in wl.ctx_lens], device=device)
    out = torch.stack([rope(q[b:b + 1], pos[b:b + 1])[0] for b in range(wl.batch)])
    return out.to(torch.float16)
