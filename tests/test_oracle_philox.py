"""Pins of the oracle's Philox4x32-10 and of the uniform mapping.

The generator is pinned against an independent implementation: cuRAND's
host-side Philox4_32_10 generator (it runs on the CPU, no GPU needed). Its
n-th block of four outputs is Philox4x32-10 with key (seed lo, seed hi) and
counter (0, 0, n, 0).
"""
import ctypes
import os

import numpy as np
import pytest

pytestmark = pytest.mark.filterwarnings("ignore")


def _curand():
    for path in ("/usr/local/cuda/lib64/libcurand.so", "libcurand.so", "libcurand.so.10"):
        try:
            return ctypes.CDLL(path)
        except OSError:
            continue
    return None


CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161


@pytest.mark.parametrize("seed", [0, 1, 1234, 0x123456789ABCDEF, 2**64 - 1])
def test_philox_matches_curand_host_generator(orc, seed):
    lib = _curand()
    if lib is None:
        pytest.skip("cuRAND not available")
    gen = ctypes.c_void_p()
    assert lib.curandCreateGeneratorHost(ctypes.byref(gen), CURAND_RNG_PSEUDO_PHILOX4_32_10) == 0
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        n_blocks = 64
        out = np.zeros(4 * n_blocks, np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(out.size)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for n in range(n_blocks):
        np.testing.assert_array_equal(orc.philox4x32_10([0, 0, n, 0], key), out[4 * n:4 * n + 4])


def test_uniform_mapping_is_open_interval_and_exact(orc):
    us = np.array([orc.uniform(7, i, j, s, p, r, w)
                   for i in range(4) for j in range(3) for s in range(3) for p in range(2)
                   for r in range(2) for w in range(4)])
    assert np.all(us > 0.0) and np.all(us < 1.0)
    # u = (2k+1) * 2^-24 for an integer k: exact in binary32
    k2 = us * 2.0**24
    np.testing.assert_array_equal(k2, np.round(k2))
    assert np.all(np.round(k2) % 2 == 1)
    np.testing.assert_array_equal(us.astype(np.float32).astype(np.float64), us)


def test_uniform_word_selection_follows_counter_layout(orc):
    seed = 99
    key = [seed & 0xFFFFFFFF, seed >> 32]
    block = orc.philox4x32_10([5, 3, 11, 1 + 4 * 2], key)
    for w in range(4):
        expect = ((int(block[w]) >> 9) + 0.5) / 2.0**23
        assert orc.uniform(seed, 5, 3, 11, 1, 2, w) == expect


def test_uniform_moments(orc):
    us = np.array([orc.uniform(3, i, 0, 0, 1, 0, w) for i in range(2500) for w in range(4)])
    assert abs(us.mean() - 0.5) < 4 * np.sqrt(1 / 12 / us.size)
    assert abs(us.var() - 1 / 12) < 0.01
