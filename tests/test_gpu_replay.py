"""Partition replay (Supp. A.8): HASH_REPLAY subspaces recompute membership from the
partition seed inside the kernels.  Their perturb / restore / commit / init / update must
match the oracle over the oracle's hash lists, leave every other element untouched, and
equal the INDICES path bit for bit (the per-element arithmetic is the same)."""
import numpy as np
import pytest
import torch

import oracle
from tolerances import assert_bf16_close, assert_perturb_fp32_close, assert_update_close

pytestmark = pytest.mark.gpu

# several hash tiles per tensor, ragged tensor ends, a tensor shorter than one group
NUMEL = [50_000, 333, 16_384, 16_385, 3, 40_000, 100_003]
TIDS = [10, 11, 12, 13, 14, 15, 16]
PSEED = 1088


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


@pytest.fixture(scope="module")
def layout(copes):
    return copes.Layout(NUMEL, TIDS)


def theta_np(n, seed=0):
    return (np.random.default_rng(seed).standard_normal(n) * 0.02).astype(np.float32)


def canary(n, dtype, seed=9):
    rng = np.random.default_rng(seed)
    if dtype == torch.bfloat16:
        b = (rng.standard_normal(n).astype(np.float32) * 0.05).view(np.uint32) >> 16
        return torch.from_numpy(b.astype(np.int16)).view(torch.bfloat16)
    return torch.from_numpy((rng.standard_normal(n) * 0.05).astype(np.float32))


def make(copes, dtype, theta):
    return copes.Arena(canary(theta.size, dtype).cuda(), torch.from_numpy(theta.copy()).cuda())


def w_bits(arena):
    if arena.w.dtype == torch.bfloat16:
        return arena.w.view(torch.int16).cpu().numpy().view(np.uint16)
    return arena.w.cpu().numpy()


def list_handle(copes, g):
    return copes.SubspaceHandle(copes.SUBSPACE_INDICES, torch.from_numpy(g.astype(np.int64)).cuda(), g.size)


def test_member_counts_match_the_oracle(copes, layout):
    for K in (1, 5, 16, 64):
        subs = copes.hash_replay_partition(layout, K, PSEED)
        assert [s.numel for s in subs] == [oracle.hash_list(NUMEL, TIDS, K, PSEED, k).size for k in range(K)]
        assert all(s.struct().K == K and s.struct().k == k for k, s in enumerate(subs))


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("K,k", [(1, 0), (4, 3), (16, 5), (64, 63)])
def test_perturb_restore_parity(copes, layout, dtype, K, k):
    n = layout.d_pad
    theta = theta_np(n)
    arena = make(copes, dtype, theta)
    twin = make(copes, dtype, theta)
    before = w_bits(arena).copy()
    sub = copes.hash_replay_partition(layout, K, PSEED, count=False)[k]
    g = oracle.hash_list(NUMEL, TIDS, K, PSEED, k).astype(np.uint64)
    inside = np.zeros(n, bool)
    inside[g] = True
    lst = list_handle(copes, g)
    for seed, ss in [(11, 2e-3), (2**40 + 5, -1e-3)]:
        copes.perturb(arena, sub, seed, ss)
        copes.perturb(twin, lst, seed, ss)
        got = w_bits(arena)
        assert np.array_equal(got, w_bits(twin))
        assert np.array_equal(got[~inside], before[~inside])
        if dtype == torch.bfloat16:
            ref_bits, _ = oracle.perturb_at(g, theta[g], seed, ss, oracle.BF16)
            scale = np.maximum(np.abs(theta[g]), np.abs(np.float32(ss) * oracle.noise(seed, g)))
            assert_bf16_close(got[g], ref_bits.astype(np.uint16), scale)
        else:
            _, exact = oracle.perturb_at(g, theta[g], seed, ss, oracle.FP32)
            assert_perturb_fp32_close(got[g], exact, theta[g], np.float32(ss) * oracle.noise(seed, g))
    copes.restore(arena, sub)
    got = w_bits(arena)
    ref = oracle.bf16_bits_array(theta[g]) if dtype == torch.bfloat16 else theta[g]
    assert np.array_equal(got[g], ref)
    assert np.array_equal(got[~inside], before[~inside])
    assert np.array_equal(arena.master.cpu().numpy(), theta)
    copes.check()


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("K,k,n_members,pairing", [(16, 2, 32, 1), (16, 15, 64, 1), (3, 1, 5, 0),
                                                    (64, 7, 256, 0), (1, 0, 8, 1)])
def test_update_parity(copes, layout, dtype, K, k, n_members, pairing):
    n = layout.d_pad
    theta = theta_np(n, seed=K + n_members)
    arena = make(copes, dtype, theta)
    twin = make(copes, dtype, theta)
    before = w_bits(arena).copy()
    sub = copes.hash_replay_partition(layout, K, PSEED, count=False)[k]
    g = oracle.hash_list(NUMEL, TIDS, K, PSEED, k).astype(np.uint64)
    inside = np.zeros(n, bool)
    inside[g] = True
    rewards = (np.random.default_rng(n_members).integers(0, 17, n_members) / 16).astype(np.float32)
    nid, sign, P = copes.member_table(n_members, pairing)
    seeds = copes.member_seeds(33, 1, k, P)
    coef = float(np.float32(5e-4 / (n_members * 1e-3)))
    f = copes.shape_fitness(torch.from_numpy(rewards).cuda(), copes.SHAPE_ZSCORE)
    copes.update(arena, sub, nid, sign, f, seeds, coef)
    copes.update(twin, list_handle(copes, g), nid, sign, f, seeds, coef)
    got = arena.master.cpu().numpy()
    assert np.array_equal(got.view(np.uint32), twin.master.cpu().numpy().view(np.uint32))
    f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(g, theta[g], seeds, wj, np.float32(coef))
    assert_update_close(got[g], exact, scale)
    assert np.array_equal(got[~inside], theta[~inside])
    wb = w_bits(arena)
    ref = oracle.bf16_bits_array(got[g]) if dtype == torch.bfloat16 else got[g]
    assert np.array_equal(wb[g], ref)
    assert np.array_equal(wb[~inside], before[~inside])
    copes.check()


def test_update_without_commit_and_init(copes, layout):
    n = layout.d_pad
    theta = theta_np(n, seed=3)
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    sub = copes.hash_replay_partition(layout, 16, PSEED, count=False)[9]
    g = oracle.hash_list(NUMEL, TIDS, 16, PSEED, 9).astype(np.uint64)
    inside = np.zeros(n, bool)
    inside[g] = True
    nid, sign, P = copes.member_table(16, copes.ANTITHETIC)
    f = torch.linspace(-1, 1, 16, device="cuda")
    copes.update(arena, sub, nid, sign, f, copes.member_seeds(33, 0, 9, P), 0.01, fuse_commit=False)
    assert np.array_equal(w_bits(arena), before)
    assert not np.array_equal(arena.master.cpu().numpy()[g], theta[g])
    copes.context_commit(arena, sub)
    wb = w_bits(arena)
    assert np.array_equal(wb[g], oracle.bf16_bits_array(arena.master.cpu().numpy()[g]))
    assert np.array_equal(wb[~inside], before[~inside])
    # synthetic init over the replayed members equals the gather path's
    twin = make(copes, torch.bfloat16, theta)
    copes.init_normal(arena, sub, 5, 0.0, 0.02)
    copes.init_normal(twin, list_handle(copes, g), 5, 0.0, 0.02)
    m1, m2 = arena.master.cpu().numpy(), twin.master.cpu().numpy()
    assert np.array_equal(m1[g].view(np.uint32), m2[g].view(np.uint32))
    assert np.array_equal(w_bits(arena)[g], w_bits(twin)[g])
    copes.check()


def test_table_past_the_arena_is_skipped_and_reported(copes, layout):
    """A replay table whose tensors run past n_alloc: the kernels skip those tiles (no
    access outside the arena) and copes_check reports the device range check."""
    theta = theta_np(60_000)
    arena = make(copes, torch.bfloat16, theta)
    before = w_bits(arena).copy()
    sub = copes.hash_replay_partition(layout, 4, PSEED, count=False)[0]  # d_pad > 60,000
    copes.perturb(arena, sub, 1, 1e-3)
    with pytest.raises(copes.CopesError) as e:
        copes.check()
    assert e.value.code == copes.ERR_DEVICE_CHECK
    got = w_bits(arena)
    g = oracle.hash_list(NUMEL, TIDS, 4, PSEED, 0)
    # tiles wholly inside the arena were processed; nothing outside the members changed
    outside = np.ones(60_000, bool)
    outside[g[g < 60_000]] = False
    assert np.array_equal(got[outside], before[outside])
    copes.check()


@pytest.mark.parametrize("K,k", [(1, 0), (16, 5), (64, 63), (3, 2)])
def test_membership_mask_equals_hashing(copes, layout, K, k):
    """A replay subspace with its membership mask gives the hashing path's results bit for
    bit: perturb, restore, update (fused commit)."""
    n = layout.d_pad
    theta = theta_np(n, seed=K)
    a1, a2 = make(copes, torch.bfloat16, theta), make(copes, torch.bfloat16, theta)
    s1 = copes.hash_replay_partition(layout, K, PSEED, count=False)[k]
    s2 = copes.hash_replay_partition(layout, K, PSEED, count=False)[k]
    mask = copes.hash_replay_mask(a2, s2)
    # the mask holds exactly the oracle's members
    bits = np.unpackbits(mask.cpu().numpy().view(np.uint8), bitorder="little").astype(bool)
    assert bits.sum() == oracle.hash_list(NUMEL, TIDS, K, PSEED, k).size
    for seed, ss in [(3, 1e-3), (4, -2e-3)]:
        copes.perturb(a1, s1, seed, ss)
        copes.perturb(a2, s2, seed, ss)
        assert np.array_equal(w_bits(a1), w_bits(a2))
    copes.restore(a1, s1)
    copes.restore(a2, s2)
    nid, sign, P = copes.member_table(32, copes.ANTITHETIC)
    f = torch.linspace(-1, 1, 32, device="cuda")
    seeds = copes.member_seeds(33, 0, k, P)
    copes.update(a1, s1, nid, sign, f, seeds, 0.2)
    copes.update(a2, s2, nid, sign, f, seeds, 0.2)
    assert np.array_equal(w_bits(a1), w_bits(a2))
    assert torch.equal(a1.master.view(torch.int32), a2.master.view(torch.int32))
    copes.drop_replay_mask(s2)
    copes.perturb(a2, s2, 5, 1e-3)
    copes.perturb(a1, s1, 5, 1e-3)
    assert np.array_equal(w_bits(a1), w_bits(a2))
    copes.check()
