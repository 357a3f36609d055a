"""Pins for oracle.philox: NVIDIA cuRAND's host Philox4x32-10 generator (a
library, run on the CPU), the dither grid, uniformity and stream
uniqueness."""

import ctypes
import ctypes.util
import os

import numpy as np
import pytest

from oracle import philox

CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161


def _curand():
    for name in ("/usr/local/cuda/lib64/libcurand.so", ctypes.util.find_library("curand")):
        if name and (os.path.exists(name) or not name.startswith("/")):
            try:
                return ctypes.CDLL(name)
            except OSError:
                pass
    return None


def _curand_block(lib, seed, block):
    """Words 4*block .. 4*block+3 of cuRAND's host Philox stream."""
    gen = ctypes.c_void_p()
    if lib.curandCreateGeneratorHost(ctypes.byref(gen), CURAND_RNG_PSEUDO_PHILOX4_32_10) != 0:
        pytest.skip("cuRAND host generator unavailable")
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        assert lib.curandSetGeneratorOffset(gen, ctypes.c_ulonglong(4 * block)) == 0
        buf = np.zeros(4, dtype=np.uint32)
        assert lib.curandGenerate(gen, buf.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(4)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    return buf


def test_philox_matches_curand_host_generator():
    """cuRAND's host generator interleaves 65536 subsequences: block B of
    its output is Philox4x32-10 at counter (B >> 16, B >> 48, B & 0xFFFF, 0)
    under key (seed lo, seed hi) (established by experiment; it exercises
    both key words and counter words 0-2)."""
    lib = _curand()
    if lib is None:
        pytest.skip("libcurand not found")
    rng = np.random.default_rng(20)
    seeds = [0, 1, 0xDEADBEEF12345678] + [int(x) for x in rng.integers(0, 2 ** 63, 3)]
    blocks = [0, 1, 65535, 65536, 123456789, (1 << 48) + (7 << 16) + 9]
    blocks += [int(x) for x in rng.integers(0, 2 ** 60, 4)]
    for seed in seeds:
        for B in blocks:
            ctr = np.array([[(B >> 16) & 0xFFFFFFFF, (B >> 48) & 0xFFFFFFFF, B & 0xFFFF, 0]], np.uint64)
            want = _curand_block(lib, seed, B)
            got = philox.philox4x32(ctr, (seed & 0xFFFFFFFF, seed >> 32))[0]
            assert np.array_equal(got, want), (seed, B)


@pytest.mark.parametrize("bits", [8, 10])
def test_dither_grid_and_uniformity(bits):
    j = philox.dither_integers(7, 3, 1, np.arange(20000), 0, 128, bits)
    assert j.min() >= 0 and j.max() < (1 << bits)
    xi = philox.dither_values(j, bits)
    assert np.all(xi >= -0.5) and np.all(xi < 0.5)
    assert np.all((xi * (1 << (bits + 1))) % 2 == 1)             # odd / 2^(bits+1)
    n = j.size
    counts = np.bincount(j.reshape(-1), minlength=1 << bits)
    chi2 = np.sum((counts - n / (1 << bits)) ** 2 / (n / (1 << bits)))
    dof = (1 << bits) - 1
    assert abs(chi2 - dof) < 6 * np.sqrt(2 * dof)
    assert abs(xi.mean()) < 5 * np.sqrt(1 / 12 / n)
    assert xi.var() == pytest.approx(1 / 12 - 1 / (12 * (1 << bits) ** 2), rel=0.01)
    # channels are not correlated with each other
    corr = np.corrcoef(xi[:, :16].T)
    assert np.max(np.abs(corr - np.eye(16))) < 0.05


def test_streams_are_distinct():
    base = dict(seed=5, layer=2, kv_head=1, tag=0)
    ref = philox.dither_integers(5, 2, 1, np.arange(64), 0, 128, 8)
    variants = [
        philox.dither_integers(6, 2, 1, np.arange(64), 0, 128, 8),
        philox.dither_integers(5 + (1 << 32), 2, 1, np.arange(64), 0, 128, 8),
        philox.dither_integers(5, 3, 1, np.arange(64), 0, 128, 8),
        philox.dither_integers(5, 2, 0, np.arange(64), 0, 128, 8),
        philox.dither_integers(5, 2, 1, np.arange(64), 1, 128, 8),
        philox.dither_integers(5, 2, 1, np.arange(64, 128), 0, 128, 8),
    ]
    for v in variants:
        assert np.mean(v == ref) < 0.02
    assert base
    # channel groups within one slot are distinct streams
    assert np.mean(ref[:, :16] == ref[:, 16:32]) < 0.02


def test_channel_word_layout():
    """Channel i of a call is byte i%4 of word i//4 (8-bit) or bits
    16*(i%2).. of word i//2 (10-bit), counter (slot, layer<<16|head, group, tag)."""
    seed, layer, head, slot = 0x1234_5678_9ABC, 4, 3, 777
    words = philox.philox4x32(np.array([[slot, layer * 65536 + head, 5, 1]], np.uint64),
                              (seed & 0xFFFFFFFF, seed >> 32))[0]
    j8 = philox.dither_integers(seed, layer, head, np.array([slot]), 1, 128, 8)[0]
    assert j8[5 * 16 + 6] == (int(words[1]) >> 16) & 0xFF
    j10 = philox.dither_integers(seed, layer, head, np.array([slot]), 1, 128, 10)[0]
    assert j10[5 * 8 + 3] == (int(words[1]) >> 16) & 0x3FF
