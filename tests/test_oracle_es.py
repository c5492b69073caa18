"""Pins for the oracle's ES steps (CPU only): rounding, perturb / restore, shaping, the
update, seeds and step sizes.  Each pin ties the oracle to a library routine, a closed
form, an invariant stated by the paper, a value the paper prints, or a statistical bound.
"""
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
from scipy import stats

import oracle
import philox_bigint

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def paper_values():
    vals = {}
    with open(os.path.join(GOLDEN, "paper_values.txt")) as fh:
        for line in fh:
            line = line.split("#")[0].strip()
            if line:
                k, v = line.split()
                vals[k] = float(v)
    return vals


# --------------------------------------------------------------------------- rounding
def test_bf16_rounding_matches_torch_for_fp32_inputs():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * 0.02,
        rng.standard_normal(2000).astype(np.float32) * 1e30,
        rng.standard_normal(2000).astype(np.float32) * 1e-39,  # fp32/bf16 subnormals
        # exact ties: the bit pattern with the dropped half equal to 0x8000
        (np.arange(4000, dtype=np.uint32) * 977 << 16 | 0x8000).view(np.float32),
    ]).astype(np.float32)
    x = x[np.isfinite(x)]
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.bf16_bits_array(x.astype(np.float64))
    assert np.array_equal(got, ref)


def exact_bf16_bits(x: float) -> int:
    """Round-half-even of a double to bf16 with Python rationals (normal range only)."""
    if x == 0:
        return 0x8000 if np.signbit(x) else 0
    f = Fraction(x)
    sign = f < 0
    a = -f if sign else f
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    quantum = Fraction(2) ** (e - 7)
    q = a / quantum
    n = q.numerator // q.denominator
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    v = float(n * quantum) * (-1 if sign else 1)
    return int(np.array([v], dtype=np.float32).view(np.uint32)[0] >> 16)


def test_bf16_rounding_of_fp64_values_is_single_rounding():
    rng = np.random.default_rng(1)
    base = rng.standard_normal(3000) * 0.05
    # values a hair above / below bf16 midpoints, where double rounding via fp32 would fail
    mids = []
    for v in base[:500]:
        b = exact_bf16_bits(v)
        lo = np.array([b << 16], dtype=np.uint32).view(np.float32)[0]
        hi = np.array([(b + 1) << 16], dtype=np.uint32).view(np.float32)[0]
        mid = (float(lo) + float(hi)) / 2
        mids += [mid, np.nextafter(mid, 0), np.nextafter(mid, 1), mid + 2.0**-40 * abs(mid)]
    for v in list(base) + mids:
        assert oracle.bf16_bits(v) == exact_bf16_bits(v), v


# ------------------------------------------------------------------------------ perturb
def _rand_master(n, seed=0):
    return (np.random.default_rng(seed).standard_normal(n) * 0.02).astype(np.float32)


def _bf16_of(master):
    return torch.from_numpy(master).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()


@pytest.mark.parametrize("kind", ["ranges", "indices"])
def test_perturb_restore_roundtrip_and_outside_untouched(kind):
    n = 4096
    master = _rand_master(n)
    w0 = _bf16_of(master)
    w0[100] ^= 0x0001  # an element outside S that does not equal round(theta)
    if kind == "ranges":
        sub = oracle.make_subspace(ranges=[(5, 700), (1024, 1030), (2000, 3001)])
        inside = np.zeros(n, bool)
        for b, e in [(5, 700), (1024, 1030), (2000, 3001)]:
            inside[b:e] = True
    else:
        idx = np.sort(np.random.default_rng(2).choice(n, 900, replace=False)).astype(np.int64)
        idx = idx[idx != 100]
        sub = oracle.make_subspace(indices=idx)
        inside = np.zeros(n, bool)
        inside[idx] = True
    w = w0.copy()
    oracle.perturb(w, master, sub, seed=77, signed_sigma=1e-3)
    assert np.array_equal(w[~inside], w0[~inside])
    assert np.mean(w[inside] != w0[inside]) > 0.5  # sigma/theta ~ 0.05: most bf16 values move
    oracle.restore(w, master, sub)
    expect = w0.copy()
    expect[inside] = _bf16_of(master)[inside]
    assert np.array_equal(w, expect)


def test_perturb_fp32_working_tensor_and_symmetry():
    n = 2048
    master = _rand_master(n, 4)
    g = np.arange(n, dtype=np.uint64)
    bits_p, ex_p = oracle.perturb_at(g, master, 9, 1e-3, oracle.FP32)
    bits_m, ex_m = oracle.perturb_at(g, master, 9, -1e-3, oracle.FP32)
    # antithetic pair symmetric about theta before rounding (each fp64 sum rounds once)
    ulp = np.spacing(np.maximum(np.abs(ex_p), np.abs(ex_m)))
    assert np.all(np.abs((ex_p - master) + (ex_m - master)) <= 2 * ulp)
    got = bits_p.view(np.float32)
    assert np.array_equal(got, ex_p.astype(np.float32))
    # the perturbation has the requested scale: (w - theta)/sigma ~ N(0, 1)
    z = (ex_p - master.astype(np.float64)) / np.float64(np.float32(1e-3))
    assert abs(z.mean()) < 5 / np.sqrt(n) and abs(z.std() - 1) < 5 * np.sqrt(0.5 / n)
    # and it is exactly the noise vector scaled: z == eps
    assert np.allclose(z, oracle.noise(9, g), rtol=1e-9, atol=1e-12)


def test_perturb_is_idempotent_from_master():
    n = 1024
    master = _rand_master(n, 5)
    sub = oracle.make_subspace(ranges=[(0, n)])
    w1 = _bf16_of(master)
    oracle.perturb(w1, master, sub, 3, 2e-3)
    w2 = w1.copy()
    oracle.perturb(w2, master, sub, 3, 2e-3)
    assert np.array_equal(w1, w2)


# ------------------------------------------------------------------------------ shaping
def test_zscore_matches_scipy_and_closed_forms():
    rng = np.random.default_rng(0)
    for n in (2, 3, 8, 40, 64, 128):
        r = rng.random(n).astype(np.float32)
        f = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE)
        ref = stats.zscore(r.astype(np.float64), ddof=0)
        assert np.allclose(f, ref, rtol=1e-6, atol=1e-7)
        assert abs(f.astype(np.float64).mean()) < 1e-6
        assert abs((f.astype(np.float64) ** 2).mean() - 1.0) < 1e-5  # population variance 1
    assert list(oracle.shape_fitness(np.array([0, 1], np.float32), oracle.SHAPE_ZSCORE)) == [-1.0, 1.0]
    f = oracle.shape_fitness(np.array([1, 2, 3], np.float32), oracle.SHAPE_ZSCORE)
    assert np.allclose(f, [-np.sqrt(1.5), 0.0, np.sqrt(1.5)], rtol=1e-7)
    # equal rewards: zero fitness (zero update), no NaN
    for v in (0.0, 0.1, 0.5625):
        assert np.all(oracle.shape_fitness(np.full(32, v, np.float32), oracle.SHAPE_ZSCORE) == 0.0)


def test_grouped_zscore_is_per_group_and_reduces_to_joint_for_one_group():
    rng = np.random.default_rng(1)
    r = rng.random(40).astype(np.float32)
    group = np.repeat(np.arange(4), 10).astype(np.int32)
    f = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE_GROUPED, group)
    for k in range(4):
        sel = group == k
        assert np.allclose(f[sel], stats.zscore(r[sel].astype(np.float64)), rtol=1e-6, atol=1e-7)
    one = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE_GROUPED, np.zeros(40, np.int32))
    assert np.array_equal(one, oracle.shape_fitness(r, oracle.SHAPE_ZSCORE))
    # a group with all-equal rewards gets zero fitness while the others do not
    r2 = r.copy()
    r2[group == 2] = 0.25
    f2 = oracle.shape_fitness(r2, oracle.SHAPE_ZSCORE_GROUPED, group)
    assert np.all(f2[group == 2] == 0) and np.all(f2[group == 0] == f[group == 0])


def test_centered_rank_matches_scipy_rankdata():
    rng = np.random.default_rng(2)
    for n in (2, 5, 16, 33, 128):
        r = (rng.integers(0, 9, size=n) / 8).astype(np.float32)  # many ties, like Bernoulli means
        f = oracle.shape_fitness(r, oracle.SHAPE_CENTERED_RANK)
        rank1 = stats.rankdata(r, method="average").astype(np.float64)  # 1-based average ranks
        ref = (rank1 - 1) / (n - 1) - 0.5
        assert np.array_equal(f, ref.astype(np.float32))
    r = np.arange(10, dtype=np.float32)[::-1].copy()
    assert np.allclose(oracle.shape_fitness(r, oracle.SHAPE_CENTERED_RANK),
                       np.linspace(0.5, -0.5, 10), atol=1e-7)
    assert np.all(oracle.shape_fitness(np.full(7, 0.3, np.float32), oracle.SHAPE_CENTERED_RANK) == 0)
    assert oracle.shape_fitness(np.array([0.7], np.float32), oracle.SHAPE_CENTERED_RANK)[0] == 0


def test_shape_none_is_identity():
    r = np.random.default_rng(3).random(16).astype(np.float32)
    assert np.array_equal(oracle.shape_fitness(r, oracle.SHAPE_NONE), r)


# ----------------------------------------------------------------------- seeds / scales
def test_member_table_and_seeds():
    nid, sign, P = oracle.member_table(8, oracle.ANTITHETIC)
    assert P == 4 and list(nid) == [0, 0, 1, 1, 2, 2, 3, 3] and list(sign) == [1, -1] * 4
    nid, sign, P = oracle.member_table(5, oracle.ONE_SIDED)
    assert P == 5 and list(nid) == list(range(5)) and list(sign) == [1] * 5
    for it, k, j in [(0, 0, 0), (3, 7, 15), (10**6, 3, 63)]:
        w = philox_bigint.philox((j, k, it, oracle.TAG_SEED), (33, 0))
        assert oracle.member_seed(33, it, k, j) == w[0] | (w[1] << 32)


def test_sigma_k_printed_value_and_step_coefficients():
    pv = paper_values()
    d = 4_659_865_088
    K = int(pv["K"])
    assert int(pv["N"]) // K == int(pv["N_k"])
    s = oracle.sigma_eff(pv["sigma"], d, d / K, True)
    assert abs(s - pv["sigma_k"]) <= 1e-15
    assert oracle.sigma_eff(1e-3, d, d / 4, False) == 1e-3
    assert oracle.step_coef(5e-4, 10, 2e-3, oracle.COEF_PAPER) == 5e-4 / 10
    assert oracle.step_coef(5e-4, 32, 1e-3, oracle.COEF_OPENAI) == 5e-4 / (32 * 1e-3)


# ------------------------------------------------------------------------------- update
def _seeds(P, base=33, it=0, k=0):
    return np.array([oracle.member_seed(base, it, k, j) for j in range(P)], dtype=np.uint64)


def test_equal_rewards_give_zero_update_bit_exact():
    n = 3000
    master = _rand_master(n, 6)
    before = master.copy()
    sub = oracle.make_subspace(ranges=[(0, n)])
    nid, sign, P = oracle.member_table(16, oracle.ANTITHETIC)
    for mode in (oracle.SHAPE_ZSCORE, oracle.SHAPE_CENTERED_RANK):
        f = oracle.shape_fitness(np.full(16, 0.375, np.float32), mode)
        oracle.update(master, sub, nid, sign, f, _seeds(P), 0.0156)
        assert np.array_equal(master.view(np.uint32), before.view(np.uint32))


def test_one_hot_update_is_the_scaled_noise_vector():
    n = 2500
    master = _rand_master(n, 7)
    sub = oracle.make_subspace(ranges=[(0, n)])
    nid, sign, P = oracle.member_table(8, oracle.ANTITHETIC)
    seeds = _seeds(P)
    alpha, N, sigma = 5e-4, 8, 1e-3
    for convention in (oracle.COEF_OPENAI, oracle.COEF_PAPER):
        c = np.float32(oracle.step_coef(alpha, N, sigma, convention))
        for m in (0, 5):
            f = np.zeros(8, np.float32)
            f[m] = 1.0
            f = oracle.shape_fitness(f, oracle.SHAPE_NONE)
            th = master.copy()
            oracle.update(th, sub, nid, sign, f, seeds, c)
            eps = oracle.noise(int(seeds[nid[m]]), np.arange(n))
            expect = (master.astype(np.float64) + float(c) * sign[m] * eps).astype(np.float32)
            assert np.array_equal(th, expect)


def test_update_outside_subspace_untouched_and_commit():
    n = 4096
    master = _rand_master(n, 8)
    w = _bf16_of(master)
    ranges = [(64, 1000), (3000, 3100)]
    sub = oracle.make_subspace(ranges=ranges)
    inside = np.zeros(n, bool)
    for b, e in ranges:
        inside[b:e] = True
    nid, sign, P = oracle.member_table(8, oracle.ANTITHETIC)
    f = oracle.shape_fitness(np.random.default_rng(0).random(8).astype(np.float32), oracle.SHAPE_ZSCORE)
    th = master.copy()
    w2 = w.copy()
    oracle.update(th, sub, nid, sign, f, _seeds(P), np.float32(0.0625), w=w2)
    assert np.array_equal(th[~inside], master[~inside]) and np.array_equal(w2[~inside], w[~inside])
    assert np.all(th[inside] != master[inside])
    assert np.array_equal(w2[inside], _bf16_of(th)[inside])


def test_k1_one_sided_paper_convention_is_standard_es():
    """Eq. 6 with N one-sided directions, population z-scores and alpha / N, rebuilt with
    numpy/scipy: theta+ = theta + (alpha/N) E^T zscore(r)."""
    n, N, alpha = 500, 12, 5e-4
    master = _rand_master(n, 9)
    r = np.random.default_rng(9).random(N).astype(np.float32)
    nid, sign, P = oracle.member_table(N, oracle.ONE_SIDED)
    seeds = _seeds(P, it=4)
    f = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE)
    c = np.float32(oracle.step_coef(alpha, N, 1e-3, oracle.COEF_PAPER))
    th = master.copy()
    oracle.update(th, oracle.make_subspace(ranges=[(0, n)]), nid, sign, f, seeds, c)
    E = np.stack([oracle.noise(int(s), np.arange(n)) for s in seeds])  # [N, n]
    rhat = stats.zscore(r.astype(np.float64), ddof=0)
    assert np.allclose(f, rhat, rtol=1e-6, atol=1e-7)
    # the update consumes the stored fp32 fitness; with those inputs the result is the
    # fp64 value rounded once, so it lies within one fp32 ulp of it
    ref = master.astype(np.float64) + np.float64(c) * (E.T @ f.astype(np.float64))
    assert np.all(np.abs(th - ref) <= np.spacing(np.abs(ref).astype(np.float32)))


def test_synchronous_composition_equals_sum_of_subspace_updates():
    """Eq. 13 / Algorithm 1: all subspace estimates come from the same pre-update theta,
    and disjoint supports make the composed update the sum of the per-subspace ones."""
    n, K = 4000, 4
    master = _rand_master(n, 10)
    parts = [[(k * n // K, (k + 1) * n // K)] for k in range(K)]
    N_k = 6
    rng = np.random.default_rng(10)
    r = rng.random(K * N_k).astype(np.float32)
    f_all = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE)  # joint standardisation
    nid, sign, P = oracle.member_table(N_k, oracle.ANTITHETIC)
    composed = master.copy()
    delta = np.zeros(n, np.float64)
    for k in range(K):
        seeds = _seeds(P, k=k)
        f = f_all[k * N_k:(k + 1) * N_k]
        oracle.update(composed, oracle.make_subspace(ranges=parts[k]), nid, sign, f, seeds,
                      np.float32(5e-4 / N_k))
        alone = master.copy()
        oracle.update(alone, oracle.make_subspace(ranges=parts[k]), nid, sign, f, seeds,
                      np.float32(5e-4 / N_k))
        delta += alone.astype(np.float64) - master
    assert np.array_equal(composed, (master.astype(np.float64) + delta).astype(np.float32))


def test_synchronous_composed_update_rebuilt_with_numpy():
    """Eq. 12 + Eq. 13 written out as linear algebra: joint z-scores over all K N_k rewards
    (scipy), then theta+ = theta + sum_k (alpha / N_k) P_k E_k^T (s * f_k), with E_k the
    member directions (antithetic: member 2j is +eps_j, 2j+1 is -eps_j) and P_k the
    restriction to S_k (Eq. 8), each S_k's directions from its own seeds.  The oracle's
    composed step lies within one fp32 ulp of that fp64 value."""
    n, K, N_k, alpha = 1200, 3, 8, 5e-4
    master = _rand_master(n, 12)
    bounds = [0, 300, 700, n]  # unequal subspaces
    r = np.random.default_rng(12).random(K * N_k).astype(np.float32)
    f_all = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE)
    assert np.allclose(f_all, stats.zscore(r.astype(np.float64), ddof=0), rtol=1e-6, atol=1e-7)
    nid, sign, P = oracle.member_table(N_k, oracle.ANTITHETIC)
    th = master.copy()
    ref = master.astype(np.float64)
    for k in range(K):
        lo, hi = bounds[k], bounds[k + 1]
        seeds = _seeds(P, k=k)
        f = f_all[k * N_k:(k + 1) * N_k]
        c = np.float32(oracle.step_coef(alpha, N_k, 1e-3, oracle.COEF_PAPER))
        oracle.update(th, oracle.make_subspace(ranges=[(lo, hi)]), nid, sign, f, seeds, c)
        g = np.arange(lo, hi)
        eps = np.stack([oracle.noise(int(s), g) for s in seeds])  # [P, d_k]
        E = np.stack([(1.0 if i % 2 == 0 else -1.0) * eps[i // 2] for i in range(N_k)])  # [N_k, d_k]
        ref[lo:hi] += np.float64(c) * (E.T @ f.astype(np.float64))
    assert np.all(np.abs(th - ref) <= np.spacing(np.abs(ref).astype(np.float32)))


def test_linear_objective_estimate_converges():
    """On r(theta) = c . theta with antithetic pairs, NONE shaping and coefficient
    alpha / (N sigma), the update divided by alpha is (1/P) sum_j (c . eps_j) eps_j, whose
    mean is c and whose mean squared error is |c|^2 (d + 1) / P."""
    d, P, sigma = 64, 1 << 16, 1e-3
    N = 2 * P
    rng = np.random.default_rng(11)
    c = rng.standard_normal(d)
    master = np.zeros(d, np.float32)
    g = np.arange(d, dtype=np.uint64)
    nid, sign, _ = oracle.member_table(N, oracle.ANTITHETIC)
    seeds = _seeds(P, it=1)
    r = np.zeros(N, np.float32)
    for j in range(P):
        _, ex_p = oracle.perturb_at(g, master, int(seeds[j]), sigma, oracle.FP32)
        _, ex_m = oracle.perturb_at(g, master, int(seeds[j]), -sigma, oracle.FP32)
        r[2 * j], r[2 * j + 1] = c @ ex_p, c @ ex_m
    f = oracle.shape_fitness(r, oracle.SHAPE_NONE)
    wj = oracle.noise_weights(nid, sign, f, P)
    alpha = 1.0
    coef = np.float32(alpha / (N * np.float32(sigma)))
    est, exact, _ = oracle.update_at(g, master, seeds, wj, coef)
    ghat = exact / alpha
    err = np.sum((ghat - c) ** 2)
    assert err <= 4 * (d + 1) * np.sum(c ** 2) / P, (err, np.sum(c ** 2))
    # with z-scored rewards the direction still converges to c
    fz = oracle.shape_fitness(r, oracle.SHAPE_ZSCORE)
    _, exz, _ = oracle.update_at(g, master, seeds, oracle.noise_weights(nid, sign, fz, P), 1.0)
    cos = exz @ c / np.linalg.norm(exz) / np.linalg.norm(c)
    assert cos > 0.99
