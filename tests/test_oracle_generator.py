"""Pins for the oracle's generator and normal transform (CPU only).

Each test ties the oracle to something other than itself: published Philox4x32-10
known-answer vectors, an independent big-int Philox, cuRAND's host-side Philox run as a
black box, scipy's normal quantile, and distribution statistics.
"""
import ctypes
import ctypes.util
import os
from fractions import Fraction

import numpy as np
import pytest
from scipy import special, stats

import oracle
import philox_bigint

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def load_kat():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as fh:
        for line in fh:
            line = line.split("#")[0].strip()
            if not line:
                continue
            parts = line.split()
            assert parts[0] == "10"
            vals = [int(x, 16) for x in parts[1:]]
            rows.append((vals[0:4], vals[4:6], vals[6:10]))
    return rows


@pytest.mark.parametrize("ctr,key,expected", load_kat())
def test_philox_known_answers(ctr, key, expected):
    assert list(oracle.philox4x32_10(ctr, key)) == expected
    assert list(philox_bigint.philox(ctr, key)) == expected


def test_philox_matches_independent_bigint():
    rng = np.random.default_rng(7)
    for _ in range(500):
        ctr = [int(x) for x in rng.integers(0, 2**32, size=4, dtype=np.uint64)]
        key = [int(x) for x in rng.integers(0, 2**32, size=2, dtype=np.uint64)]
        assert tuple(int(x) for x in oracle.philox4x32_10(ctr, key)) == philox_bigint.philox(ctr, key)


def test_philox_stream_counter_layout():
    seed = 0x0123456789ABCDEF
    q0 = (1 << 33) - 3  # crosses a 32-bit carry into the counter's second word
    words = oracle.philox_stream(seed, q0, 6, aux=5, tag=oracle.TAG_PARTITION)
    for i in range(6):
        assert tuple(int(x) for x in words[i]) == philox_bigint.words(
            seed, q0 + i, aux=5, tag=oracle.TAG_PARTITION)


def _curand_host():
    path = ctypes.util.find_library("curand")
    for cand in [path, "/usr/local/cuda/lib64/libcurand.so", "libcurand.so.10"]:
        if not cand:
            continue
        try:
            return ctypes.CDLL(cand)
        except OSError:
            continue
    return None


def test_philox_matches_curand_host_generator():
    """cuRAND's CURAND_RNG_PSEUDO_PHILOX4_32_10 host generator, run as a black box:
    its output block b is Philox4x32-10 at counter (0, 0, b, 0) under key = the seed's
    two 32-bit halves (observed ordering of the library's default layout)."""
    lib = _curand_host()
    if lib is None:
        pytest.skip("libcurand not available")
    gen = ctypes.c_void_p()
    if lib.curandCreateGeneratorHost(ctypes.byref(gen), 161) != 0:
        pytest.skip("cuRAND host generator unavailable")
    try:
        seed = 0x9E3779B97F4A7C15
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        n = 4 * 256
        out = np.zeros(n, dtype=np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(n)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for b in range(256):
        assert list(out[4 * b:4 * b + 4]) == list(oracle.philox4x32_10([0, 0, b, 0], key))


def test_uniform_exact_odd_multiples():
    rng = np.random.default_rng(1)
    xs = [0, 1, 2, 255, 256, 0x7FFFFE, 0x7FFFFF, 0x800000, 0xFFFFFFFF] + [
        int(x) for x in rng.integers(0, 2**32, size=2000, dtype=np.uint64)]
    for x in xs:
        u = oracle.uniform(x)
        frac = Fraction(u) * (1 << 23)
        assert frac.denominator == 1 and frac.numerator % 2 == 1
        assert frac.numerator == ((x % (1 << 23)) | 1)  # bits 1..22 of the word, made odd
        assert 0.0 < u < 1.0
        assert np.float32(u) == u  # exact in fp32
    assert oracle.uniform(0) == 2.0**-23
    assert oracle.uniform(0xFFFFFFFF) == 1.0 - 2.0**-23
    # only bits 1..22 matter
    assert oracle.uniform(0xFF800000 | 0x1234) == oracle.uniform(0x1235)


def test_quantile_exhaustive_against_scipy():
    """All 2^22 values the transform can see, against scipy.special.ndtri."""
    m = np.arange(1 << 22, dtype=np.float64)
    u = (2.0 * m + 1.0) * 2.0**-23
    oracle.clear_fault()
    q = oracle.normal_quantile_array(u)
    assert oracle.fault_flag() == 0
    ref = special.ndtri(u)
    rel = np.abs(q - ref) / np.abs(ref)
    assert rel.max() < 1e-13, rel.max()
    # symmetry Phi^-1(u) = -Phi^-1(1 - u), exactly (1 - u is exact)
    assert np.array_equal(q, -q[::-1])
    # monotone
    assert np.all(np.diff(q) > 0)


def test_noise_composition_matches_independent_pieces():
    """eps_seed[g] = Phi^-1(u(word g&3 of Philox at counter g>>2)), rebuilt from the big-int
    Philox and scipy's quantile."""
    seed = 12345678901234567
    rng = np.random.default_rng(3)
    g = np.concatenate([np.arange(0, 16), rng.integers(0, 2**40, size=300)]).astype(np.uint64)
    eps = oracle.noise(seed, g)
    for gi, e in zip(g.tolist(), eps.tolist()):
        w = philox_bigint.words(seed, gi >> 2)[gi & 3]
        u = ((w & 0x7FFFFE) | 1) * 2.0**-23
        assert abs(e - special.ndtri(u)) <= 1e-13 * max(1.0, abs(e))


def test_noise_distribution_statistics():
    n = 1 << 22
    x = oracle.noise_range(2024, 0, n)
    se = 1.0 / np.sqrt(n)
    assert abs(x.mean()) < 5 * se
    assert abs(x.var() - 1.0) < 5 * np.sqrt(2.0 / n)
    assert abs(stats.skew(x)) < 5 * np.sqrt(6.0 / n)
    assert abs(stats.kurtosis(x)) < 5 * np.sqrt(24.0 / n)
    ks = stats.kstest(x, "norm")
    assert ks.pvalue > 1e-3
    # a second seed and the init tag are independent streams
    y = oracle.noise_range(2025, 0, n)
    z = oracle.noise_range(2024, 0, n, tag=oracle.TAG_INIT)
    assert abs(np.corrcoef(x, y)[0, 1]) < 5 * se
    assert abs(np.corrcoef(x, z)[0, 1]) < 5 * se
    # neighbouring elements (same Philox block, and across blocks) are uncorrelated
    assert abs(np.corrcoef(x[:-1], x[1:])[0, 1]) < 5 * se
    assert abs(np.corrcoef(x[:-4], x[4:])[0, 1]) < 5 * se
