"""Parity at the workloads' full sizes, in the launch configuration the benchmark times.

The oracle computes sampled outputs element by element. Samples include every subspace
range's first and last elements and random interior ones. Inputs come from seeded
generators: numpy for the tiny vector, torch's seeded CUDA generator for the large
arenas. The rewards are seeded synthetic scalars shared by both sides. Size-independent
properties are checked on the whole subspace: restore is exact, and elements outside S
are untouched.
"""
import gc

import numpy as np
import pytest
import torch

import oracle
from paper_2608_02391_gb300 import workloads as wl
from tolerances import (assert_bf16_close, assert_fitness_close, assert_perturb_fp32_close,
                        assert_update_close)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


@pytest.fixture(autouse=True)
def free_memory():
    yield
    gc.collect()
    torch.cuda.empty_cache()


SHAPE = {"zscore": oracle.SHAPE_ZSCORE, "centered_rank": oracle.SHAPE_CENTERED_RANK,
         "zscore_grouped": oracle.SHAPE_ZSCORE_GROUPED, "none": oracle.SHAPE_NONE}


def make_arena(copes, w: wl.Workload, seed=0):
    """fp32 master ~ N(0, 0.02^2) from torch's seeded CUDA generator, norms = 1.0, and
    w = bf16(master)."""
    layout = copes.Layout(w.numel)
    master = torch.empty(layout.d_pad, dtype=torch.float32, device="cuda")
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed)
    master.normal_(0.0, w.init_scale, generator=gen)
    off = layout.offsets
    for t, ten in enumerate(w.tensors):
        if ten.kind == "norm":
            master[int(off[t]):int(off[t]) + ten.numel].fill_(1.0)
    return copes.Arena(master.to(torch.bfloat16), master), layout


def sample_from_ranges(ranges, n_random, rng):
    edges = []
    for b, e in ranges:
        edges += [b, min(b + 1, e - 1), max(e - 2, b), e - 1]
    sizes = np.array([e - b for b, e in ranges], dtype=np.float64)
    pick = rng.choice(len(ranges), size=n_random, p=sizes / sizes.sum())
    rnd = [int(ranges[i][0] + rng.integers(0, ranges[i][1] - ranges[i][0])) for i in pick]
    return np.unique(np.array(edges + rnd, dtype=np.int64))


def tile_ranges(sub):
    t = sub.tensor.cpu().numpy()
    out = []
    for b, e in t:
        if out and out[-1][1] == int(b):
            out[-1] = (out[-1][0], int(e))
        else:
            out.append((int(b), int(e)))
    return out


def bf16_bits_of(t: torch.Tensor, idx: np.ndarray):
    return t.view(torch.int16)[torch.from_numpy(idx).cuda()].cpu().numpy().view(np.uint16)


def check_visit(copes, arena, sub, sample, w: wl.Workload, k, iteration, rewards, pairing=None,
                check_members=(0, 1)):
    """One round-robin visit on the GPU; the oracle recomputes the sampled outputs."""
    pairing = copes.ANTITHETIC if pairing is None else pairing
    N = w.n_members
    nid, sign, P = copes.member_table(N, pairing)
    seeds = copes.member_seeds(w.base_seed, iteration, k, P)
    sigma = np.float32(w.sigma)
    idx_t = torch.from_numpy(sample).cuda()
    theta = arena.master[idx_t].cpu().numpy()
    g = sample.astype(np.uint64)
    w_outside_sum = None
    for i in range(N):
        copes.perturb(arena, sub, int(seeds[nid[i]]), float(sign[i] * sigma))
        if i in check_members:
            ref_bits, _ = oracle.perturb_at(g, theta, int(seeds[nid[i]]), float(sign[i] * sigma), oracle.BF16)
            scale = np.maximum(np.abs(theta), np.abs(sigma * oracle.noise(int(seeds[nid[i]]), g)))
            assert_bf16_close(bf16_bits_of(arena.w, sample), ref_bits.astype(np.uint16), scale)
    copes.restore(arena, sub)
    assert np.array_equal(bf16_bits_of(arena.w, sample), oracle.bf16_bits_array(theta))
    r_dev = torch.from_numpy(rewards).cuda()
    f = copes.shape_fitness(r_dev, w.shaping).cpu().numpy()
    f_ref = oracle.shape_fitness(rewards, SHAPE[w.shaping])
    assert_fitness_close(f, f_ref)
    coef = np.float32(copes.step_coef(w.alpha, N, float(sigma), copes.COEF_OPENAI))
    copes.update(arena, sub, nid, sign, torch.from_numpy(f).cuda(), seeds, float(coef), fuse_commit=True)
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(g, theta, seeds, wj, coef)
    got = arena.master[idx_t].cpu().numpy()
    assert_update_close(got, exact, scale)
    assert np.array_equal(bf16_bits_of(arena.w, sample), oracle.bf16_bits_array(got))


def whole_subspace_properties(copes, arena, sub, seed):
    """Restore after perturb is exact on all of S; elements outside S keep their bits."""
    before = arena.w.view(torch.int16).clone()
    copes.perturb(arena, sub, seed, 1e-3)
    copes.restore(arena, sub)
    assert torch.equal(arena.w.view(torch.int16), before)
    del before


# ------------------------------------------------------------------------------ tiny
def test_tiny_round_robin_loop_matches_oracle_trajectory(copes):
    """The tiny workload end to end: 3 cycles x 4 contiguous subspaces x 8 antithetic
    members, rewards r_i = c . w_i computed by the oracle from its own perturbed weights.
    GPU and oracle run independent trajectories from the same rewards. Errors add across a
    subspace's 3 updates, so the tolerance is the sum of the per-update bounds."""
    w = wl.workload("tiny")
    theta0, cvec = wl.tiny_theta_and_objective()
    n = theta0.size
    K, N = w.K, w.n_members
    sigma = np.float32(w.sigma)
    coef = np.float32(w.alpha / (N * float(sigma)))
    o_master = theta0.copy()
    bound = np.zeros(n)
    g_master = torch.from_numpy(theta0.copy()).cuda()
    arena = copes.Arena(g_master.clone(), g_master)  # fp32 working tensor
    layout = copes.Layout([n])
    nid, sign, P = oracle.member_table(N, oracle.ANTITHETIC)
    for cycle in range(w.cycles):
        for k in range(K):
            ranges = oracle.contiguous_ranges([n], K, k)
            (b, e), = ranges
            sub = copes.subspace_build(layout, copes.PART_CONTIGUOUS, K, k, tile_size=1 << 14)
            assert tile_ranges(sub) == ranges
            seeds = np.array([oracle.member_seed(w.base_seed, cycle, k, j) for j in range(P)], np.uint64)
            g = np.arange(b, e, dtype=np.uint64)
            rewards = np.zeros(N, np.float32)
            base_dot = float(cvec @ o_master) - float(cvec[b:e] @ o_master[b:e])
            for i in range(N):
                _, exact = oracle.perturb_at(g, o_master[b:e], int(seeds[nid[i]]), float(sign[i] * sigma), oracle.FP32)
                rewards[i] = np.float32(base_dot + float(cvec[b:e] @ exact))
                copes.perturb(arena, sub, int(seeds[nid[i]]), float(sign[i] * sigma))
                if i == 0:
                    got = arena.w[b:e].cpu().numpy()
                    ref_theta = o_master[b:e]
                    eps = oracle.noise(int(seeds[nid[i]]), g)
                    # the GPU perturbs its own master, which differs from the oracle's by the
                    # bound accumulated so far
                    tol = 1e-6 * np.maximum.reduce([np.abs(exact), np.abs(ref_theta), np.abs(sigma * eps)]) + bound[b:e]
                    assert np.all(np.abs(got - exact) <= tol)
            copes.restore(arena, sub)
            f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
            f = copes.shape_fitness(torch.from_numpy(rewards).cuda(), "zscore")
            assert_fitness_close(f.cpu().numpy(), f_ref)
            copes.update(arena, sub, nid, sign, f, seeds, float(coef), fuse_commit=True)
            wj = oracle.noise_weights(nid, sign, f_ref, P)
            _, exact, scale = oracle.update_at(g, o_master[b:e], seeds, wj, coef)
            o_master[b:e] = exact.astype(np.float32)
            bound[b:e] += 1e-6 * np.maximum(np.abs(exact), scale)
            got = g_master[b:e].cpu().numpy()
            assert np.all(np.abs(got.astype(np.float64) - exact) <= bound[b:e])
            assert torch.equal(arena.w[b:e], g_master[b:e])  # fp32 commit is a copy
    copes.check()


# ------------------------------------------------------------------------ 0.5B / 4B / 8B
@pytest.mark.parametrize("name,visits", [("0.5b", range(8)), ("4b", [0, 3, 7])])
def test_layer_block_workloads_sampled(copes, name, visits):
    w = wl.workload(name)
    arena, layout = make_arena(copes, w)
    rng = np.random.default_rng(5)
    rewards = wl.reward_stream(w, 8)
    for k in visits:
        sub = copes.subspace_build(layout, copes.PART_TENSOR_GROUPS, w.K, k, group_of=w.group_of,
                                   tile_size=copes.DEFAULT_TILE)
        ranges = tile_ranges(sub)
        assert ranges == oracle.group_ranges(w.numel, w.group_of, k)
        sample = sample_from_ranges(ranges, 4096, rng)
        check_visit(copes, arena, sub, sample, w, k, 0, rewards[k])
        if k == visits[0]:
            whole_subspace_properties(copes, arena, sub, 99)
    copes.check()


@pytest.mark.parametrize("name", ["0.5b", "4b"])
def test_visits_on_four_working_copies_as_benched(copes, name):
    """The bench's configuration of the layer-block workloads: tile tables of 16,384
    elements, members written two
    pairs at a time into four working copies (es.round_robin_visit with
    Partner.four_copies), restore, shaping and the fused update + commit to every copy.
    Every member's live weights, the update and the commit are checked against the oracle
    on sampled indices of the first and last layer blocks; after each visit the four
    copies are bit-identical."""
    from paper_2608_02391_gb300 import es
    w = wl.workload(name)
    arena1, layout = make_arena(copes, w)
    arena = copes.Arena(arena1.w, arena1.master, *[arena1.w.clone() for _ in range(3)])
    partner = es.Partner.four_copies(arena)
    cfg = es.ESConfig(n_members=w.n_members, sigma=w.sigma, alpha=w.alpha, shaping=w.shaping)
    nid, sign, P = copes.member_table(w.n_members, copes.ANTITHETIC)
    rewards = wl.reward_stream(w, 8)
    rng = np.random.default_rng(9)
    for k in (0, w.K - 1):
        sub = copes.subspace_build(layout, copes.PART_TENSOR_GROUPS, w.K, k, group_of=w.group_of,
                                   tile_size=copes.DEFAULT_TILE)
        sample = sample_from_ranges(tile_ranges(sub), 2048, rng)
        idx_t = torch.from_numpy(sample).cuda()
        theta = arena.master[idx_t].cpu().numpy()
        g = sample.astype(np.uint64)
        seeds = copes.member_seeds(cfg.base_seed, 0, k, P)
        s_k64 = es.sigma_k(cfg, layout.d_pad, sub.numel)  # the visit's sigma_k (a double)
        s_k = float(np.float32(s_k64))  # as the kernels receive it
        live = {}

        def evaluate(i):  # the live copy's bits at the sample, as a rollout would read them
            live[i] = arena.live.view(torch.int16)[idx_t].cpu().numpy().view(np.uint16)

        r_dev = torch.from_numpy(rewards[k]).cuda()
        f = es.round_robin_visit(arena, sub, k, 0, cfg, layout.d_pad, r_dev, evaluate=evaluate, partner=partner)
        copes.check()
        assert sorted(live) == list(range(w.n_members))
        for i in range(w.n_members):
            seed, s = int(seeds[nid[i]]), float(sign[i]) * s_k
            ref_bits, _ = oracle.perturb_at(g, theta, seed, s, oracle.BF16)
            scale = np.maximum(np.abs(theta), np.abs(np.float32(s_k) * oracle.noise(seed, g)))
            assert_bf16_close(live[i], ref_bits.astype(np.uint16), scale)
        f_ref = oracle.shape_fitness(rewards[k], SHAPE[w.shaping])
        assert_fitness_close(f.cpu().numpy(), f_ref)
        coef = np.float32(copes.step_coef(cfg.alpha, w.n_members, s_k64, cfg.convention))
        _, exact, scale = oracle.update_at(g, theta, seeds, oracle.noise_weights(nid, sign, f_ref, P), coef)
        got = arena.master[idx_t].cpu().numpy()
        assert_update_close(got, exact, scale)
        commit = oracle.bf16_bits_array(got)
        for c in arena.copies:
            assert np.array_equal(bf16_bits_of(c, sample), commit)
            assert torch.equal(c.view(torch.int16), arena.w.view(torch.int16))


def test_8b_type_groups_sampled(copes):
    w = wl.workload("8b")
    arena, layout = make_arena(copes, w)
    rng = np.random.default_rng(8)
    rewards = wl.reward_stream(w, 4)
    for k in (0, 2):  # attention (1.51e9 parameters), norms + embeddings
        sub = copes.subspace_build(layout, copes.PART_TENSOR_GROUPS, w.K, k, group_of=w.group_of,
                                   tile_size=copes.DEFAULT_TILE)
        ranges = tile_ranges(sub)
        assert ranges == oracle.group_ranges(w.numel, w.group_of, k)
        check_visit(copes, arena, sub, sample_from_ranges(ranges, 4096, rng), w, k, 0, rewards[k],
                    check_members=(0, 127))
    copes.check()


def test_8b_full_cc_loop_sampled(copes):
    """The 8B workload as configured: 10 cooperative-coevolution cycles over the 4 type
    groups (40 visits, N = 128 antithetic), through the round-robin schedule.  After every
    visit the oracle recomputes the shaped fitness and the updated master at sampled
    members of that subspace from the values they held before it, and the commit is checked
    against the new master."""
    from paper_2608_02391_gb300 import es
    w = wl.workload("8b")
    assert w.cycles == 10
    arena, layout = make_arena(copes, w)
    rng = np.random.default_rng(10)
    subs, samples = [], []
    for k in range(w.K):
        sub = copes.subspace_build(layout, copes.PART_TENSOR_GROUPS, w.K, k, group_of=w.group_of,
                                   tile_size=copes.DEFAULT_TILE)
        subs.append(sub)
        samples.append(sample_from_ranges(tile_ranges(sub), 1024, rng))
    cfg = es.ESConfig(n_members=w.n_members, sigma=w.sigma, alpha=w.alpha, shaping=w.shaping)
    rewards = wl.reward_stream(w, w.cycles * w.K)
    nid, sign, P = copes.member_table(w.n_members, copes.ANTITHETIC)
    sigma = np.float32(w.sigma)
    coef = np.float32(copes.step_coef(w.alpha, w.n_members, float(sigma), copes.COEF_OPENAI))
    for cycle in range(w.cycles):
        for k in range(w.K):
            idx = torch.from_numpy(samples[k]).cuda()
            before = arena.master[idx].cpu().numpy()
            r = rewards[cycle * w.K + k]
            f = es.round_robin_visit(arena, subs[k], k, cycle, cfg, w.d, torch.from_numpy(r).cuda())
            f_ref = oracle.shape_fitness(r, SHAPE[w.shaping])
            assert_fitness_close(f.cpu().numpy(), f_ref)
            seeds = copes.member_seeds(w.base_seed, cycle, k, P)
            wj = oracle.noise_weights(nid, sign, f_ref, P)
            _, exact, scale = oracle.update_at(samples[k].astype(np.uint64), before, seeds, wj, coef)
            got = arena.master[idx].cpu().numpy()
            assert_update_close(got, exact, scale)
            assert np.array_equal(bf16_bits_of(arena.w, samples[k]), oracle.bf16_bits_array(got))
    copes.check()


# ---------------------------------------------------------------------------- 4B hash
def test_4b_hash_partition_and_gather_visit(copes):
    w = wl.workload("4b-hash")
    arena, layout = make_arena(copes, w)
    tids = list(range(len(w.tensors)))
    layout = copes.Layout(w.numel, tids)
    lists = copes.hash_partition(layout, w.K, w.partition_seed)
    counts = np.array([s.numel for s in lists])
    assert counts.sum() == w.d
    sd = np.sqrt(w.d / w.K * (1 - 1 / w.K))
    assert np.all(np.abs(counts - w.d / w.K) < 5 * sd)
    for s in lists:
        assert bool((s.tensor[1:] > s.tensor[:-1]).all())
    # membership of random elements, from the oracle's hash
    rng = np.random.default_rng(11)
    off = oracle.layout(w.numel)
    for _ in range(2000):
        t = int(rng.integers(0, len(w.tensors)))
        e = int(rng.integers(0, w.numel[t]))
        k = oracle.hash_subspace(w.partition_seed, tids[t], e, w.K)
        g = int(off[t]) + e
        pos = int(torch.searchsorted(lists[k].tensor, torch.tensor([g], device="cuda")).item())
        assert pos < lists[k].numel and int(lists[k].tensor[pos].item()) == g
    # one gather visit on subspace 3 with the workload's N = 64
    sub = lists[3]
    pos = np.unique(np.concatenate([[0, 1, sub.numel - 1], rng.integers(0, sub.numel, 4096)]))
    sample = sub.tensor[torch.from_numpy(pos).cuda()].cpu().numpy()
    rewards = wl.reward_stream(w, 4)[3]
    check_visit(copes, arena, sub, sample, w, 3, 0, rewards)
    del lists
    copes.check()


def test_4b_hash_replay_visit_equals_list_path(copes):
    """Partition replay at the 4B-hash size: the HASH_REPLAY subspace's visit matches the
    oracle on sampled members, and its perturb / update equal the INDICES path on the whole
    arena bit for bit."""
    w = wl.workload("4b-hash")
    arena, _ = make_arena(copes, w)
    tids = list(range(len(w.tensors)))
    layout = copes.Layout(w.numel, tids)
    k = 3
    sub = copes.hash_replay_partition(layout, w.K, w.partition_seed)[k]
    lst = copes.hash_partition(layout, w.K, w.partition_seed)[k]
    assert sub.numel == lst.numel
    nid, sign, P = copes.member_table(w.n_members, copes.ANTITHETIC)
    seeds = copes.member_seeds(w.base_seed, 0, k, P)
    # perturb: replay vs list, whole arena
    copes.perturb(arena, sub, int(seeds[5]), -1e-3)
    w_replay = arena.w.view(torch.int16).clone()
    copes.restore(arena, sub)
    copes.perturb(arena, lst, int(seeds[5]), -1e-3)
    assert torch.equal(arena.w.view(torch.int16), w_replay)
    copes.restore(arena, lst)
    del w_replay
    # update: replay vs list, whole arena
    f = torch.linspace(-1.5, 1.5, w.n_members, device="cuda")
    master0 = arena.master.clone()
    copes.update(arena, sub, nid, sign, f, seeds, 0.25)
    m_replay, w_replay = arena.master.clone(), arena.w.view(torch.int16).clone()
    arena.master.copy_(master0)
    copes.restore(arena, lst)
    copes.update(arena, lst, nid, sign, f, seeds, 0.25)
    assert torch.equal(arena.master.view(torch.int32), m_replay.view(torch.int32))
    assert torch.equal(arena.w.view(torch.int16), w_replay)
    del m_replay, w_replay
    arena.master.copy_(master0)
    copes.restore(arena, lst)
    del master0
    # a visit with the workload's N = 64 on the replay subspace, sampled against the oracle
    rng = np.random.default_rng(12)
    pos = np.unique(np.concatenate([[0, 1, lst.numel - 1], rng.integers(0, lst.numel, 4096)]))
    sample = lst.tensor[torch.from_numpy(pos).cuda()].cpu().numpy()
    del lst
    rewards = wl.reward_stream(w, 4)[k]
    check_visit(copes, arena, sub, sample, w, k, 0, rewards)
    copes.check()


def test_4b_hash_full_sweep_replay_sampled(copes):
    """The 4B-hash workload as configured: one perturb / restore / update sweep over all 16
    hash subspaces (N = 64), on replay subspaces (no index lists), each visit checked at
    sampled members against the oracle; the members are found with the oracle's hash."""
    w = wl.workload("4b-hash")
    arena, _ = make_arena(copes, w)
    tids = list(range(len(w.tensors)))
    layout = copes.Layout(w.numel, tids)
    subs = copes.hash_replay_partition(layout, w.K, w.partition_seed)
    assert sum(s.numel for s in subs) == w.d
    rng = np.random.default_rng(16)
    off = oracle.layout(w.numel)
    per_k = [[] for _ in range(w.K)]
    sizes = np.array(w.numel, dtype=np.float64)
    for t in rng.choice(len(w.tensors), size=24_000, p=sizes / sizes.sum()):
        e = int(rng.integers(0, w.numel[t]))
        per_k[oracle.hash_subspace(w.partition_seed, tids[t], e, w.K)].append(int(off[t]) + e)
    rewards = wl.reward_stream(w, w.K)
    for k in range(w.K):
        sample = np.unique(np.array(per_k[k], dtype=np.int64))
        assert sample.size > 1000
        check_visit(copes, arena, subs[k], sample, w, k, 0, rewards[k])
    copes.check()


# ----------------------------------------------------------- beyond 2^34 global indices
def test_counters_beyond_2_34(copes):
    """Tiles past global index 2^34 take the kernels' general counter path; a range
    crossing the boundary checks both paths against the oracle."""
    n = (1 << 34) + (1 << 20)
    master = torch.empty(n, dtype=torch.float32, device="cuda")
    lo, hi = (1 << 34) - (1 << 19), (1 << 34) + (1 << 19)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(3)
    master[lo:hi].normal_(0.0, 0.02, generator=gen)
    wt = torch.zeros(n, dtype=torch.bfloat16, device="cuda")
    arena = copes.Arena(wt, master)
    sub = copes.tiles_from_ranges([(lo, hi)], tile_size=1 << 16)
    w = wl.Workload("big", [wl.Tensor("x", n, "vector")], K=1, mode="contiguous", n_members=8,
                    sigma=1e-3, alpha=5e-4, shaping="zscore")
    rng = np.random.default_rng(4)
    sample = np.unique(np.concatenate([[lo, (1 << 34) - 1, 1 << 34, hi - 1],
                                       rng.integers(lo, hi, 4000)])).astype(np.int64)
    rewards = (rng.integers(0, 17, 8) / 16).astype(np.float32)
    check_visit(copes, arena, sub, sample, w, 0, 0, rewards)
    # the antithetic pair perturb on both counter paths equals two perturbs, bit for bit
    buf = torch.empty(hi - lo, dtype=torch.bfloat16, device="cuda")
    copes.perturb(arena, sub, 77, 1e-3)
    plus = arena.w[lo:hi].view(torch.int16).clone()
    copes.perturb(arena, sub, 77, -1e-3)
    minus = arena.w[lo:hi].view(torch.int16).clone()
    copes.perturb_pair(arena, sub, 77, 1e-3, buf, lo)
    assert torch.equal(arena.w[lo:hi].view(torch.int16), plus)
    assert torch.equal(buf.view(torch.int16), minus)
    # ... and both members agree with the oracle on the sampled indices, on both sides of 2^34
    theta = arena.master[torch.from_numpy(sample).cuda()].cpu().numpy()
    g = sample.astype(np.uint64)
    scale = np.maximum(np.abs(theta), np.abs(np.float32(1e-3) * oracle.noise(77, g)))
    for s_sign, got in ((1.0, bf16_bits_of(arena.w, sample)), (-1.0, bf16_bits_of(buf, sample - lo))):
        ref_bits, _ = oracle.perturb_at(g, theta, 77, s_sign * 1e-3, oracle.BF16)
        assert_bf16_close(got, ref_bits.astype(np.uint16), scale)
    copes.check()


def test_two_pairs_beyond_2_34(copes):
    """The two-pairs perturb on a range crossing global index 2^34 (its general counter
    path above, its folded-Philox path below): each of the four working copies equals a
    plain perturb bit for bit, and agrees with the oracle on sampled indices on both
    sides.  Four bf16 copies and the fp32 master of 2^34 + 2^20 elements: 192 GB."""
    n = (1 << 34) + (1 << 20)
    lo, hi = (1 << 34) - (1 << 19), (1 << 34) + (1 << 19)
    master = torch.empty(n, dtype=torch.float32, device="cuda")
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    master[lo:hi].normal_(0.0, 0.02, generator=gen)
    copies = [torch.zeros(n, dtype=torch.bfloat16, device="cuda") for _ in range(4)]
    sub = copes.tiles_from_ranges([(lo, hi)], tile_size=1 << 16)
    members = [(77, 1e-3), (77, -1e-3), (78, 1e-3), (78, -1e-3)]
    copes.perturb_two_pairs(copes.Arena(copies[0], master, *copies[1:]), sub, 77, 78, 1e-3)
    got = [c[lo:hi].view(torch.int16).clone() for c in copies]
    del copies[1:]
    single = copes.Arena(copies[0], master)
    rng = np.random.default_rng(6)
    sample = np.unique(np.concatenate([[lo, (1 << 34) - 1, 1 << 34, hi - 1],
                                       rng.integers(lo, hi, 4000)])).astype(np.int64)
    theta = master[torch.from_numpy(sample).cuda()].cpu().numpy()
    g = sample.astype(np.uint64)
    for c, (seed, s) in enumerate(members):
        copes.perturb(single, sub, seed, s)
        assert torch.equal(copies[0][lo:hi].view(torch.int16), got[c]), c
        scale = np.maximum(np.abs(theta), np.abs(np.float32(s) * oracle.noise(seed, g)))
        ref_bits, _ = oracle.perturb_at(g, theta, seed, s, oracle.BF16)
        mine = got[c][torch.from_numpy(sample - lo).cuda()].cpu().numpy().view(np.uint16)
        assert_bf16_close(mine, ref_bits.astype(np.uint16), scale)
    copes.check()


# ------------------------------------------------------------------ Algorithm 1 (SYNC)
@pytest.mark.parametrize("joint", [True, False])
def test_sync_step_algorithm1_matches_oracle(copes, joint):
    """Algorithm 1 on a 1M-parameter vector: a random equal-size chunk partition, K = 4,
    N = 8 (N_k = 2), sigma_k = sqrt(K) sigma (Eq. 11), joint (Eq. 12) or per-subspace
    standardisation, coefficient alpha / N_k (Eq. 13), every g_k from the same
    pre-update theta."""
    from paper_2608_02391_gb300 import es
    n, K, N, chunk = 1 << 20, 4, 8, 4096
    theta0, _ = wl.tiny_theta_and_objective()
    master = torch.from_numpy(theta0.copy()).cuda()
    arena = copes.Arena(master.to(torch.bfloat16), master)
    layout = copes.Layout([n])
    subs = es.build_subspaces(layout, "random_chunks", K, seed=77, chunk=chunk)
    cmap = oracle.random_chunks(n // chunk, K, 77)
    for k in range(K):
        assert tile_ranges(subs[k]) == oracle.chunk_ranges([n], chunk, cmap, k)
    cfg = es.ESConfig(n_members=N, sigma=1e-3, alpha=5e-4, shaping="zscore",
                      convention=copes.COEF_PAPER, dimension_aware=True)
    rewards = (np.random.default_rng(2).integers(0, 17, N) / 16).astype(np.float32)
    f = es.sync_step(arena, subs, 0, cfg, n, torch.from_numpy(rewards).cuda(), joint=joint)
    group = np.repeat(np.arange(K), N // K).astype(np.int32)
    f_ref = (oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE) if joint
             else oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE_GROUPED, group))
    assert_fitness_close(f.cpu().numpy(), f_ref)
    nid, sign, P = oracle.member_table(N // K, oracle.ANTITHETIC)
    got = master.cpu().numpy()
    for k in range(K):
        ranges = oracle.chunk_ranges([n], chunk, cmap, k)
        g = np.concatenate([np.arange(b, e) for b, e in ranges]).astype(np.uint64)
        s_k = oracle.sigma_eff(1e-3, n, g.size, True)
        assert abs(s_k - 2e-3) < 1e-18  # sqrt(K) sigma with K = 4 (Sec. 4.1)
        seeds = np.array([oracle.member_seed(33, 0, k, j) for j in range(P)], np.uint64)
        coef = np.float32(oracle.step_coef(5e-4, N // K, s_k, oracle.COEF_PAPER))
        wj = oracle.noise_weights(nid, sign, f_ref[k * (N // K):(k + 1) * (N // K)], P)
        _, exact, scale = oracle.update_at(g, theta0[g.astype(np.int64)], seeds, wj, coef)
        assert_update_close(got[g.astype(np.int64)], exact, scale)
    copes.check()


def test_sync_steps_with_prefetched_partitions_are_bit_identical(copes):
    """Algorithm 1 resamples the partition every step.  Building step s + 1's partition on
    a side stream while step s runs (es.ChunkPrefetcher) gives the oracle's chunk ranges and
    the same three-step trajectory, bit for bit, as building each partition in line."""
    from paper_2608_02391_gb300 import es
    n, K, N, chunk, steps = 1 << 20, 4, 8, 4096, 3
    theta0, _ = wl.tiny_theta_and_objective()
    layout = copes.Layout([n])
    cfg = es.ESConfig(n_members=N, sigma=1e-3, alpha=5e-4, shaping="zscore",
                      convention=copes.COEF_PAPER, dimension_aware=True)
    rewards = torch.from_numpy((np.random.default_rng(3).integers(0, 17, (steps, N)) / 16)
                               .astype(np.float32)).cuda()
    seed_of = lambda s: 500 + s  # noqa: E731

    def run(prefetch):
        master = torch.from_numpy(theta0.copy()).cuda()
        arena = copes.Arena(master.to(torch.bfloat16), master)
        parts = es.ChunkPrefetcher(layout, K, seed_of, chunk=chunk)
        seen = []
        for s in range(steps):
            if prefetch:
                subs = parts.take(s)
            else:
                subs = es.build_subspaces(layout, "random_chunks", K, seed=seed_of(s), chunk=chunk)
            seen.append([tile_ranges(sub) for sub in subs])
            es.sync_step(arena, subs, s, cfg, n, rewards[s], joint=True)
            if prefetch and s + 1 < steps:
                parts.prefetch(s + 1)
        torch.cuda.synchronize()
        return master.cpu().numpy(), arena.w.view(torch.int16).cpu().numpy(), seen

    m_ref, w_ref, seen_ref = run(False)
    m_got, w_got, seen_got = run(True)
    for s in range(steps):
        cmap = oracle.random_chunks(n // chunk, K, seed_of(s))
        for k in range(K):
            assert seen_got[s][k] == seen_ref[s][k] == oracle.chunk_ranges([n], chunk, cmap, k)
    assert np.array_equal(m_got.view(np.uint32), m_ref.view(np.uint32))
    assert np.array_equal(w_got, w_ref)
    assert not np.array_equal(m_ref, theta0)
    copes.check()
