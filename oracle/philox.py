"""Philox4x32-10 and the subtractive dither derived from it.

Test infrastructure only (see ``oracle/__init__.py``).

The paper draws the dither with Philox4x32-10 (Salmon, Moraes, Dror, Shaw,
"Parallel random numbers: as easy as 1, 2, 3", SC'11) from a counter built
from (layer, KV head, slot, channel) so that the read side can regenerate
exactly the dither used at write time (§6.2.1 "Research kernels and the
proof--kernel contract"; §6.2.3 "The dither counter uses the slot, not the
sequence position").  The paper fixes the generator and the tuple but not
the word layout; the reading used here (shared with the CUDA path only as
a written definition) is:

  key     = (seed mod 2^32, seed >> 32)
  counter = (slot, layer * 2^16 + kv_head, channel_group, tag)   tag 0 = K, 1 = V
  each call yields 128 bits; with ``bits`` = 8 one call covers 16 channels
  (channel i of the group = byte i%4 of word i//4), with ``bits`` = 10 one
  call covers 8 channels (channel i = bits [16*(i%2), 16*(i%2)+10) of word
  i//2).  The integer j in [0, 2^bits) maps to the dither
  xi = (j + 1/2) / 2^bits - 1/2, a midpoint grid on [-1/2, 1/2) whose mean is
  exactly 0 (§4.2 "Subtractive dither": xi ~ U[-1/2, 1/2)).
"""

import numpy as np

M0 = np.uint64(0xD2511F53)
M1 = np.uint64(0xCD9E8D57)
W0 = 0x9E3779B9
W1 = 0xBB67AE85
MASK32 = np.uint64(0xFFFFFFFF)
ROUNDS = 10


def philox4x32(counter, key, rounds=ROUNDS):
    """Philox4x32 bijection.

    counter: uint32 array [..., 4]; key: two uint32 scalars or arrays
    broadcastable to counter[..., 0].  Returns uint32 [..., 4].
    """
    c = np.asarray(counter, dtype=np.uint64) & MASK32
    c0, c1, c2, c3 = c[..., 0], c[..., 1], c[..., 2], c[..., 3]
    k0 = np.asarray(key[0], dtype=np.uint64) & MASK32
    k1 = np.asarray(key[1], dtype=np.uint64) & MASK32
    for r in range(rounds):
        if r > 0:                                   # key schedule (Weyl bump)
            k0 = (k0 + np.uint64(W0)) & MASK32
            k1 = (k1 + np.uint64(W1)) & MASK32
        p0 = M0 * c0                                # 32x32 -> 64-bit products
        p1 = M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def channels_per_call(bits):
    if bits == 8:
        return 16
    if bits == 10:
        return 8
    raise ValueError("dither_bits must be 8 or 10")


def dither_integers(seed, layer, kv_head, slots, tag, head_dim, bits):
    """Integer dither j[slot, channel] in [0, 2^bits) for the given slots.

    slots: int array [n]; returns int64 [n, head_dim].
    """
    slots = np.asarray(slots, dtype=np.int64)
    per_call = channels_per_call(bits)
    n_groups = head_dim // per_call
    n = slots.shape[0]
    ctr = np.zeros((n, n_groups, 4), dtype=np.uint64)
    ctr[..., 0] = slots[:, None].astype(np.uint64)
    ctr[..., 1] = np.uint64(layer * 65536 + kv_head)
    ctr[..., 2] = np.arange(n_groups, dtype=np.uint64)[None, :]
    ctr[..., 3] = np.uint64(tag)
    key = (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    words = philox4x32(ctr, key).astype(np.int64)          # [n, groups, 4]
    i = np.arange(per_call)
    if bits == 8:
        j = (words[..., i // 4] >> (8 * (i % 4))) & 0xFF
    else:
        j = (words[..., i // 2] >> (16 * (i % 2))) & 0x3FF
    return j.reshape(n, head_dim)


def dither_values(j, bits):
    """Dither xi = (j + 1/2) / 2^bits - 1/2 (exact in float64)."""
    return (np.asarray(j, dtype=np.float64) + 0.5) / float(1 << bits) - 0.5
