"""CPU weight backup mode (bf16 weights on the GPU, the context as a bf16 copy in pinned
host memory, no fp32 master): save, perturb, restore and update against the oracle with
theta = the backup's values, untouched elements outside S on both copies, and the same
results as the master path when the master holds the backup's values."""
import numpy as np
import pytest
import torch

import oracle
from tolerances import assert_bf16_close

pytestmark = pytest.mark.gpu

N_ALLOC = 60_000
RANGES = [(3, 9_001), (9_001, 9_003), (12_345, 30_000), (30_064, 30_065), (40_001, 59_997)]


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


def bf16_canary(n, seed, scale=0.05):
    b = (np.random.default_rng(seed).standard_normal(n).astype(np.float32) * scale).view(np.uint32) >> 16
    return torch.from_numpy(b.astype(np.uint16).view(np.int16)).view(torch.bfloat16)


def bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def as_f32(b):
    return (b.astype(np.uint32) << 16).view(np.float32)


def make(copes, seed_w=1, seed_b=2):
    w = bf16_canary(N_ALLOC, seed_w).cuda()
    backup = bf16_canary(N_ALLOC, seed_b, 0.02).pin_memory()
    return copes.BackupArena(w, backup)


def inside_mask():
    m = np.zeros(N_ALLOC, bool)
    for b, e in RANGES:
        m[b:e] = True
    return m


@pytest.mark.parametrize("tile", [4096, 999])
def test_save_perturb_restore(copes, tile):
    arena = make(copes)
    sub = copes.tiles_from_ranges(RANGES, tile_size=tile)
    inside = inside_mask()
    g = np.nonzero(inside)[0].astype(np.uint64)
    w0, b0 = bits(arena.w).copy(), bits(arena.backup).copy()
    copes.backup_save(arena, sub)
    torch.cuda.synchronize()
    b1 = bits(arena.backup)
    assert np.array_equal(b1[inside], w0[inside]) and np.array_equal(b1[~inside], b0[~inside])
    theta = as_f32(b1)
    for seed, ss in [(11, 2e-3), (2**40 + 5, -1e-3)]:
        copes.backup_perturb(arena, sub, seed, ss)
        got = bits(arena.w)
        ref, _ = oracle.perturb_at(g, theta[inside], seed, ss, oracle.BF16)
        scale = np.maximum(np.abs(theta[inside]), np.abs(np.float32(ss) * oracle.noise(seed, g)))
        assert_bf16_close(got[inside], ref.astype(np.uint16), scale)
        assert np.array_equal(got[~inside], w0[~inside])
    torch.cuda.synchronize()
    assert np.array_equal(bits(arena.backup), b1)  # perturb never writes the backup
    copes.backup_restore(arena, sub)
    got = bits(arena.w)
    assert np.array_equal(got[inside], b1[inside]) and np.array_equal(got[~inside], w0[~inside])
    copes.check()


@pytest.mark.parametrize("n_members,pairing", [(32, 1), (5, 0)])
def test_update_against_oracle_and_master_path(copes, n_members, pairing):
    arena = make(copes, 3, 4)
    sub = copes.tiles_from_ranges(RANGES, tile_size=4096)
    inside = inside_mask()
    g = np.nonzero(inside)[0].astype(np.uint64)
    w0, b0 = bits(arena.w).copy(), bits(arena.backup).copy()
    theta = as_f32(b0)
    # the master path on the same context: master = backup's values
    twin = copes.Arena(arena.w.clone(), torch.from_numpy(theta.copy()).cuda())
    rewards = (np.random.default_rng(n_members).integers(0, 17, n_members) / 16).astype(np.float32)
    nid, sign, P = copes.member_table(n_members, pairing)
    seeds = copes.member_seeds(33, 2, 1, P)
    coef = float(np.float32(0.25))
    f = copes.shape_fitness(torch.from_numpy(rewards).cuda(), copes.SHAPE_ZSCORE)
    copes.backup_update(arena, sub, nid, sign, f, seeds, coef)
    copes.update(twin, sub, nid, sign, f, seeds, coef, fuse_commit=True)
    torch.cuda.synchronize()
    wb, bb = bits(arena.w), bits(arena.backup)
    assert np.array_equal(wb[inside], bb[inside])  # the new context is in both copies
    assert np.array_equal(wb[~inside], w0[~inside]) and np.array_equal(bb[~inside], b0[~inside])
    assert np.array_equal(wb[inside], bits(twin.w)[inside])  # same fp32 arithmetic as the master path
    f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(g, theta[inside], seeds, wj, np.float32(coef))
    ref = oracle.bf16_bits_array(exact.astype(np.float32))
    assert_bf16_close(wb[inside], ref, np.maximum(np.abs(exact), scale))
    copes.check()


def test_pageable_backup_is_rejected(copes):
    w = torch.zeros(1024, dtype=torch.bfloat16, device="cuda")
    backup = torch.zeros(1024, dtype=torch.bfloat16)  # not page-locked
    arena = copes.BackupArena(w, backup)
    sub = copes.tiles_from_ranges([(0, 1024)], tile_size=256)
    with pytest.raises(copes.CopesError) as e:
        copes.backup_save(arena, sub)
    assert e.value.code == copes.ERR_INVALID_ARG


@pytest.mark.parametrize("tile", [4096, 999])
def test_pair_perturb_from_the_backup(copes, tile):
    """copes_backup_perturb_pair: w as backup_perturb(+s sigma), the device partner buffer
    as backup_perturb(-s sigma), bit for bit; the partner copy then gives the second
    member; the backup and everything outside S stay untouched."""
    ref, arena = make(copes), make(copes)
    sub = copes.tiles_from_ranges(RANGES, tile_size=tile)
    inside = inside_mask()
    g = np.nonzero(inside)[0]
    for a in (ref, arena):
        copes.backup_save(a, sub)
    torch.cuda.synchronize()
    b0 = bits(arena.backup).copy()
    buf = bf16_canary(N_ALLOC, 4).cuda()
    buf0 = bits(buf).copy()
    copes.backup_perturb(ref, sub, 21, 2e-3)
    plus = bits(ref.w).copy()
    copes.backup_perturb(ref, sub, 21, -2e-3)
    minus = bits(ref.w).copy()
    copes.backup_perturb_pair(arena, sub, 21, 2e-3, buf, 0)
    assert np.array_equal(bits(arena.w), plus)
    pb = bits(buf)
    assert np.array_equal(pb[g], minus[inside])
    out = np.ones(buf.numel(), bool)
    out[g] = False
    assert np.array_equal(pb[out], buf0[out])
    copes.backup_perturb_partner(arena, sub, buf, 0)
    assert np.array_equal(bits(arena.w), minus)
    torch.cuda.synchronize()
    assert np.array_equal(bits(arena.backup), b0)
    copes.check()


def test_backup_visit_with_partner_buffer_is_bit_identical(copes):
    from paper_2608_02391_gb300 import es
    results = []
    for use in (False, True):
        arena = make(copes)
        subs = [copes.tiles_from_ranges(RANGES[:2], tile_size=4096), copes.tiles_from_ranges(RANGES[2:], tile_size=999)]
        for sub in subs:
            copes.backup_save(arena, sub)
        partners = es.Partner.per_subspace(arena, subs) if use else [None, None]
        cfg = es.ESConfig(n_members=8, sigma=1e-3, alpha=5e-4)
        rng = np.random.default_rng(2)
        trace = []
        for k, sub in enumerate(subs):
            r = torch.from_numpy(rng.standard_normal(8).astype(np.float32)).cuda()

            def ev(i):
                trace.append(int(arena.live.view(torch.int16).to(torch.int64).mul(i + 1).sum()))

            es.backup_visit(arena, sub, k, 0, cfg, N_ALLOC, r, evaluate=ev, partner=partners[k])
        torch.cuda.synchronize()
        results.append((trace, bits(arena.w).copy(), bits(arena.backup).copy()))
    copes.check()
    assert results[0][0] == results[1][0] and len(results[0][0]) == 16
    assert np.array_equal(results[0][1], results[1][1]) and np.array_equal(results[0][2], results[1][2])
