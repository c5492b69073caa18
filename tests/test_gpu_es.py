"""GPU-vs-oracle parity of the ES steps at sizes the oracle finishes in seconds: several
tiles, ragged tails, unaligned subspace edges, both working dtypes, both subspace kinds,
and the degenerate cases (empty subspaces, equal rewards, one-hot fitness)."""
import numpy as np
import pytest
import torch

import oracle
from tolerances import (assert_bf16_close, assert_fitness_close, assert_perturb_fp32_close,
                        assert_update_close)

pytestmark = pytest.mark.gpu

N_ALLOC = 60_000
RANGES = [(3, 9_001), (9_001, 9_003), (12_345, 30_000), (30_064, 30_065), (40_001, 59_997)]


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


def theta_np(n=N_ALLOC, seed=0):
    return (np.random.default_rng(seed).standard_normal(n) * 0.02).astype(np.float32)


def canary_bits(n, dtype, seed=9):
    """Random working-tensor contents, so untouched elements are recognisable."""
    rng = np.random.default_rng(seed)
    if dtype == torch.bfloat16:
        b = (rng.standard_normal(n).astype(np.float32) * 0.05).view(np.uint32) >> 16
        return torch.from_numpy(b.astype(np.int16)).view(torch.bfloat16)
    return torch.from_numpy((rng.standard_normal(n) * 0.05).astype(np.float32))


def w_bits(arena):
    if arena.w.dtype == torch.bfloat16:
        return arena.w.view(torch.int16).cpu().numpy().view(np.uint16)
    return arena.w.cpu().numpy()


def mask_of(ranges, n=N_ALLOC):
    m = np.zeros(n, bool)
    for b, e in ranges:
        m[b:e] = True
    return m


def make(copes, dtype, theta):
    master = torch.from_numpy(theta.copy()).cuda()
    w = canary_bits(theta.size, dtype).cuda()
    return copes.Arena(w, master)


def subspace(copes, kind, ranges, tile):
    if kind == "tiles":
        return copes.tiles_from_ranges(ranges, tile_size=tile)
    idx = np.concatenate([np.arange(b, e) for b, e in ranges]).astype(np.int64)
    return copes.SubspaceHandle(copes.SUBSPACE_INDICES, torch.from_numpy(idx).cuda(), idx.size)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("kind,tile", [("tiles", 4096), ("tiles", 1000), ("indices", 0)])
def test_perturb_restore_parity(copes, dtype, kind, tile):
    theta = theta_np()
    arena = make(copes, dtype, theta)
    before = w_bits(arena).copy()
    sub = subspace(copes, kind, RANGES, tile)
    inside = mask_of(RANGES)
    g = np.nonzero(inside)[0].astype(np.uint64)
    for seed, ss in [(11, 2e-3), (11, -2e-3), (2**40 + 5, 1e-3)]:
        copes.perturb(arena, sub, seed, ss)
        got = w_bits(arena)
        assert np.array_equal(got[~inside], before[~inside])
        if dtype == torch.bfloat16:
            ref_bits, _ = oracle.perturb_at(g, theta[inside], seed, ss, oracle.BF16)
            scale = np.maximum(np.abs(theta[inside]), np.abs(np.float32(ss) * oracle.noise(seed, g)))
            assert_bf16_close(got[inside], ref_bits.astype(np.uint16), scale)
        else:
            _, exact = oracle.perturb_at(g, theta[inside], seed, ss, oracle.FP32)
            eps = oracle.noise(seed, g)
            assert_perturb_fp32_close(got[inside], exact, theta[inside], np.float32(ss) * eps)
    copes.restore(arena, sub)
    got = w_bits(arena)
    if dtype == torch.bfloat16:
        ref = oracle.bf16_bits_array(theta[inside])
        assert np.array_equal(got[inside], ref)
    else:
        assert np.array_equal(got[inside], theta[inside])
    assert np.array_equal(got[~inside], before[~inside])
    copes.check()


def test_empty_subspace_is_a_no_op(copes):
    theta = theta_np(1000)
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    empty = copes.tiles_from_ranges([], tile_size=64)
    copes.perturb(arena, empty, 1, 1e-3)
    copes.restore(arena, empty)
    nid, sign, P = copes.member_table(2, copes.ANTITHETIC)
    f = torch.zeros(2, device="cuda")
    copes.update(arena, empty, nid, sign, f, copes.member_seeds(33, 0, 0, P), 0.1)
    copes.check()
    assert np.array_equal(w_bits(arena), before)
    assert np.array_equal(arena.master.cpu().numpy(), theta)


@pytest.mark.parametrize("mode", ["none", "zscore", "zscore_grouped", "centered_rank"])
@pytest.mark.parametrize("n", [1, 2, 7, 16, 32, 64, 128, 256])
def test_shape_fitness_parity(copes, mode, n):
    rng = np.random.default_rng(n)
    for r in [(rng.integers(0, 17, n) / 16).astype(np.float32), rng.random(n).astype(np.float32),
              np.full(n, 0.3125, np.float32)]:
        group = (np.arange(n) * 4 // n).astype(np.int32)
        rd = torch.from_numpy(r).cuda()
        gd = torch.from_numpy(group).cuda()
        got = copes.shape_fitness(rd, mode, gd if mode == "zscore_grouped" else None).cpu().numpy()
        ref = oracle.shape_fitness(r, copes.SHAPE_MODES[mode], group if mode == "zscore_grouped" else None)
        assert_fitness_close(got, ref)


def run_update(copes, arena, sub, rewards, pairing, mode, seeds_base, coef, fuse, n_members):
    nid, sign, P = copes.member_table(n_members, pairing)
    seeds = copes.member_seeds(seeds_base, 1, 2, P)
    rd = torch.from_numpy(rewards).cuda()
    f = copes.shape_fitness(rd, mode)
    copes.update(arena, sub, nid, sign, f, seeds, coef, fuse_commit=fuse)
    return nid, sign, P, seeds, f.cpu().numpy()


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("kind,tile", [("tiles", 4096), ("tiles", 777), ("indices", 0)])
@pytest.mark.parametrize("n_members,pairing", [(2, 1), (3, 0), (8, 1), (32, 1), (128, 1), (5, 0), (256, 0)])
def test_update_parity(copes, dtype, kind, tile, n_members, pairing):
    theta = theta_np(seed=n_members)
    arena = make(copes, dtype, theta)
    before = w_bits(arena).copy()
    sub = subspace(copes, kind, RANGES, tile)
    inside = mask_of(RANGES)
    rewards = (np.random.default_rng(n_members).integers(0, 17, n_members) / 16).astype(np.float32)
    coef = float(np.float32(5e-4 / (n_members * 1e-3)))
    nid, sign, P, seeds, f = run_update(copes, arena, sub, rewards, pairing, copes.SHAPE_ZSCORE, 33,
                                        coef, True, n_members)
    g = np.nonzero(inside)[0].astype(np.uint64)
    # the oracle shapes the same rewards itself
    f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
    assert_fitness_close(f, f_ref)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(g, theta[inside], seeds, wj, np.float32(coef))
    got = arena.master.cpu().numpy()
    assert_update_close(got[inside], exact, scale)
    assert np.array_equal(got[~inside], theta[~inside])
    wb = w_bits(arena)
    # fused commit: w = round(theta+) for the GPU's own theta+, outside untouched
    if dtype == torch.bfloat16:
        assert np.array_equal(wb[inside], oracle.bf16_bits_array(got[inside]))
    else:
        assert np.array_equal(wb[inside], got[inside])
    assert np.array_equal(wb[~inside], before[~inside])
    copes.check()


def test_update_without_commit_leaves_w(copes):
    theta = theta_np()
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    sub = subspace(copes, "tiles", RANGES, 4096)
    rewards = np.random.default_rng(1).random(16).astype(np.float32)
    run_update(copes, arena, sub, rewards, 1, copes.SHAPE_ZSCORE, 5, 0.03, False, 16)
    assert np.array_equal(w_bits(arena), before)
    copes.context_commit(arena, sub)
    inside = mask_of(RANGES)
    got = arena.master.cpu().numpy()
    assert np.array_equal(w_bits(arena)[inside], oracle.bf16_bits_array(got[inside]))


@pytest.mark.parametrize("mode", ["zscore", "centered_rank"])
def test_equal_rewards_leave_master_bit_exact(copes, mode):
    theta = theta_np()
    arena = make(copes, torch.bfloat16, theta)
    sub = subspace(copes, "tiles", RANGES, 4096)
    run_update(copes, arena, sub, np.full(32, 0.4375, np.float32), 1, copes.SHAPE_MODES[mode], 3,
               0.0156, True, 32)
    assert np.array_equal(arena.master.cpu().numpy().view(np.uint32), theta.view(np.uint32))


def test_one_hot_fitness_gives_the_noise_vector(copes):
    theta = theta_np()
    arena = make(copes, torch.float32, theta)
    sub = subspace(copes, "tiles", RANGES, 4096)
    n = 8
    nid, sign, P = copes.member_table(n, copes.ANTITHETIC)
    seeds = copes.member_seeds(33, 0, 0, P)
    f = np.zeros(n, np.float32)
    f[5] = 1.0
    coef = float(np.float32(5e-4 / (n * 1e-3)))
    copes.update(arena, sub, nid, sign, torch.from_numpy(f).cuda(), seeds, coef)
    inside = mask_of(RANGES)
    g = np.nonzero(inside)[0].astype(np.uint64)
    eps = oracle.noise(int(seeds[nid[5]]), g)
    exact = theta[inside].astype(np.float64) + np.float64(np.float32(coef)) * sign[5] * eps
    assert_update_close(arena.master.cpu().numpy()[inside], exact, np.abs(np.float32(coef) * eps))


def test_init_normal_parity(copes):
    n = 50_000
    arena = copes.Arena.empty(n, torch.bfloat16)
    sub = copes.tiles_from_ranges([(0, n)], tile_size=8192)
    copes.init_normal(arena, sub, 0, 0.0, 0.02)
    got = arena.master.cpu().numpy()
    eps = oracle.noise_range(0, 0, n, tag=oracle.TAG_INIT)
    ref = np.float64(np.float32(0.02)) * eps
    # the normal's tolerance scaled by 0.02, plus the final fp32 rounding
    assert np.all(np.abs(got - ref) <= 0.02 * 2.0**-20 * np.maximum(1.0, np.abs(eps)) + 2.0**-24 * np.abs(ref))
    assert np.array_equal(w_bits(arena), oracle.bf16_bits_array(got))


def test_device_range_checks_report_without_faulting(copes):
    theta = theta_np(1000)
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    bad_tiles = copes.SubspaceHandle(copes.SUBSPACE_TILES,
                                     torch.tensor([[0, 100], [900, 5000]], dtype=torch.int64, device="cuda"), 0)
    copes.perturb(arena, bad_tiles, 1, 1e-3)
    with pytest.raises(copes.CopesError) as e:
        copes.check()
    assert e.value.code == copes.ERR_DEVICE_CHECK
    assert np.array_equal(w_bits(arena)[100:], before[100:])  # the bad tile was skipped whole
    bad_idx = copes.SubspaceHandle(copes.SUBSPACE_INDICES,
                                   torch.tensor([5, 7, 1000, -3], dtype=torch.int64, device="cuda"), 4)
    copes.restore(arena, bad_idx)
    with pytest.raises(copes.CopesError) as e:
        copes.check()
    assert e.value.code == copes.ERR_DEVICE_CHECK
    copes.check()  # cleared


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_gathered_master_equals_master_path(copes, dtype):
    """An INDICES subspace with a gathered master: perturb, restore, update and init give
    the master path's results bit for bit, master stays untouched until the scatter, and
    the scatter publishes the gathered values."""
    theta = theta_np(seed=21)
    a1, a2 = make(copes, dtype, theta), make(copes, dtype, theta)
    s1 = subspace(copes, "indices", RANGES, 0)
    s2 = subspace(copes, "indices", RANGES, 0)
    copes.gather_master(a2, s2)
    inside = mask_of(RANGES)
    assert np.array_equal(s2.gathered.cpu().numpy(), theta[inside])
    for seed, ss in [(5, 1e-3), (6, -2e-3)]:
        copes.perturb(a1, s1, seed, ss)
        copes.perturb(a2, s2, seed, ss)
        assert np.array_equal(w_bits(a1), w_bits(a2))
    copes.restore(a1, s1)
    copes.restore(a2, s2)
    assert np.array_equal(w_bits(a1), w_bits(a2))
    nid, sign, P = copes.member_table(32, copes.ANTITHETIC)
    f = torch.linspace(-1, 1, 32, device="cuda")
    seeds = copes.member_seeds(33, 0, 1, P)
    copes.update(a1, s1, nid, sign, f, seeds, 0.3)
    copes.update(a2, s2, nid, sign, f, seeds, 0.3)
    assert np.array_equal(w_bits(a1), w_bits(a2))
    assert np.array_equal(a2.master.cpu().numpy(), theta)  # untouched until the scatter
    m1 = a1.master.cpu().numpy()
    assert np.array_equal(s2.gathered.cpu().numpy().view(np.uint32), m1[inside].view(np.uint32))
    copes.scatter_master(a2, s2)
    assert np.array_equal(a2.master.cpu().numpy().view(np.uint32), m1.view(np.uint32))
    copes.init_normal(a1, s1, 9, 0.0, 0.02)
    copes.init_normal(a2, s2, 9, 0.0, 0.02)
    assert np.array_equal(w_bits(a1), w_bits(a2))
    assert np.array_equal(s2.gathered.cpu().numpy().view(np.uint32),
                          a1.master.cpu().numpy()[inside].view(np.uint32))
    copes.check()


def test_maximum_tile_size(copes):
    """Tiles of COPES_TILE_MAX elements (the largest a tile table may hold) over a ragged
    range: perturb, restore and update against the oracle at sampled elements, with the
    range edges included; a larger tile size is rejected on the host."""
    n = (1 << 21) + 4101
    lo, hi = 3, n - 2
    theta = theta_np(n, seed=12)
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    sub = copes.tiles_from_ranges([(lo, hi)], tile_size=copes.TILE_MAX)
    assert sub.tensor.shape[0] == 3
    with pytest.raises(copes.CopesError) as e:
        copes.tiles_from_ranges([(lo, hi)], tile_size=copes.TILE_MAX + 1)
    assert e.value.code == copes.ERR_SIZE
    rng = np.random.default_rng(13)
    g = np.unique(np.concatenate([[lo, lo + 1, (1 << 20) + lo - 1, (1 << 20) + lo, hi - 2, hi - 1],
                                  rng.integers(lo, hi, 20_000)])).astype(np.uint64)
    copes.perturb(arena, sub, 77, 1.5e-3)
    got = w_bits(arena)
    ref, _ = oracle.perturb_at(g, theta[g.astype(np.int64)], 77, 1.5e-3, oracle.BF16)
    scale = np.maximum(np.abs(theta[g.astype(np.int64)]), np.abs(np.float32(1.5e-3) * oracle.noise(77, g)))
    assert_bf16_close(got[g.astype(np.int64)], ref.astype(np.uint16), scale)
    assert np.array_equal(got[:lo], before[:lo]) and np.array_equal(got[hi:], before[hi:])
    copes.restore(arena, sub)
    assert np.array_equal(w_bits(arena)[lo:hi], oracle.bf16_bits_array(theta[lo:hi]))
    nid, sign, P = copes.member_table(32, copes.ANTITHETIC)
    rewards = np.linspace(0, 1, 32).astype(np.float32)
    f = copes.shape_fitness(torch.from_numpy(rewards).cuda(), copes.SHAPE_ZSCORE)
    seeds = copes.member_seeds(33, 0, 0, P)
    copes.update(arena, sub, nid, sign, f, seeds, 0.01)
    f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scl = oracle.update_at(g, theta[g.astype(np.int64)], seeds, wj, np.float32(0.01))
    m = arena.master.cpu().numpy()
    assert_update_close(m[g.astype(np.int64)], exact, scl)
    assert np.array_equal(m[:lo], theta[:lo]) and np.array_equal(m[hi:], theta[hi:])
    copes.check()
