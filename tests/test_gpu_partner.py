"""Antithetic pair perturb (copes_perturb_pair / copes_perturb_partner) against the oracle
and against two independent perturbs, for every subspace kind and both working dtypes:
the member's weights, the partner's weights written to the buffer and then copied in, the
buffer and the weights left untouched outside S, the buffer's range check, and whole ES
visits and Algorithm 1 steps with and without the buffer."""
import numpy as np
import pytest
import torch

import oracle
from tolerances import assert_bf16_close, assert_perturb_fp32_close

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


def canary(n, dtype, seed):
    rng = np.random.default_rng(seed)
    if dtype == torch.bfloat16:
        b = (rng.standard_normal(n).astype(np.float32) * 0.05).view(np.uint32) >> 16
        return torch.from_numpy(b.astype(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy((rng.standard_normal(n) * 0.05).astype(np.float32)).cuda()


def bits(t):
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy().view(np.uint32)


def mask_of(ranges, n=N_ALLOC):
    m = np.zeros(n, bool)
    for b, e in ranges:
        m[b:e] = True
    return m


def make_sub(copes, kind, ranges, arena):
    if kind.startswith("tiles"):
        return copes.tiles_from_ranges(ranges, tile_size=int(kind.split(":")[1]))
    idx = np.concatenate([np.arange(b, e) for b, e in ranges]).astype(np.int64)
    sub = copes.SubspaceHandle(copes.SUBSPACE_INDICES, torch.from_numpy(idx).cuda(), idx.size)
    if kind == "gathered":
        sub.gathered = torch.empty(idx.size, dtype=torch.float32, device="cuda")
        copes.gather_master(arena, sub)
    return sub


def check_member(got_bits, dtype, g, theta_in, seed, ss):
    """The bits of one member's weights at g against the oracle's perturb."""
    if dtype == torch.bfloat16:
        ref_bits, _ = oracle.perturb_at(g, theta_in, seed, ss, oracle.BF16)
        scale = np.maximum(np.abs(theta_in), np.abs(np.float32(ss) * oracle.noise(seed, g)))
        assert_bf16_close(got_bits, ref_bits.astype(np.uint16), scale)
    else:
        _, exact = oracle.perturb_at(g, theta_in, seed, ss, oracle.FP32)
        assert_perturb_fp32_close(got_bits.view(np.float32), exact, theta_in,
                                  np.float32(ss) * oracle.noise(seed, g))


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("kind", ["tiles:4096", "tiles:1000", "indices", "gathered"])
@pytest.mark.parametrize("ranges,base", [(RANGES, 0), (RANGES[2:], 12_344)])
def test_pair_equals_two_perturbs_and_the_oracle(copes, dtype, kind, ranges, base):
    theta = theta_np()
    inside = mask_of(ranges)
    g = np.nonzero(inside)[0].astype(np.uint64)
    w0 = canary(N_ALLOC, dtype, 9)
    ref = copes.Arena(w0.clone(), torch.from_numpy(theta.copy()).cuda())
    arena = copes.Arena(w0.clone(), torch.from_numpy(theta.copy()).cuda())
    sub_ref, sub = make_sub(copes, kind, ranges, ref), make_sub(copes, kind, ranges, arena)
    buf = canary(N_ALLOC - base, dtype, 5)
    buf0 = bits(buf).copy()
    for seed, ss in [(11, 2e-3), (2**40 + 5, -1e-3)]:
        copes.perturb(ref, sub_ref, seed, ss)
        plus = bits(ref.w).copy()
        copes.perturb(ref, sub_ref, seed, -ss)
        minus = bits(ref.w).copy()
        copes.perturb_pair(arena, sub, seed, ss, buf, base)
        got = bits(arena.w)
        assert np.array_equal(got, plus)  # w exactly as copes_perturb(+ss), untouched outside S
        pb = bits(buf)
        assert np.array_equal(pb[g.astype(np.int64) - base], minus[inside])
        assert np.array_equal(pb[~inside[base:]], buf0[~inside[base:]])  # the buffer outside S
        check_member(pb[g.astype(np.int64) - base], dtype, g, theta[inside], seed, -ss)
        check_member(got[inside], dtype, g, theta[inside], seed, ss)
        copes.perturb_partner(arena, sub, buf, base)
        assert np.array_equal(bits(arena.w), minus)
    copes.check()


@pytest.mark.parametrize("masked", [False, True])
def test_pair_on_replayed_hash_subspaces(copes, masked):
    layout = copes.Layout([20_000, 7, 39_000])
    n = layout.d_pad
    theta = theta_np(n)
    w0 = canary(n, torch.bfloat16, 9)
    ref = copes.Arena(w0.clone(), torch.from_numpy(theta.copy()).cuda())
    arena = copes.Arena(w0.clone(), torch.from_numpy(theta.copy()).cuda())
    for k, sub in enumerate(copes.hash_replay_partition(layout, 4, 77)):
        if masked:
            copes.hash_replay_mask(arena, sub)
        buf = canary(n, torch.bfloat16, 5 + k)
        copes.perturb(ref, sub, 3 + k, 1e-3)
        plus = bits(ref.w).copy()
        copes.perturb(ref, sub, 3 + k, -1e-3)
        minus = bits(ref.w).copy()
        copes.perturb_pair(arena, sub, 3 + k, 1e-3, buf, 0)
        assert np.array_equal(bits(arena.w), plus)
        copes.perturb_partner(arena, sub, buf, 0)
        assert np.array_equal(bits(arena.w), minus)
    copes.check()


@pytest.mark.parametrize("kind", ["tiles:4096", "indices"])
def test_partner_range_is_checked_without_faulting(copes, kind):
    """A buffer range that misses part of S: the kernels skip the missing elements (whole
    tiles for TILES), write nothing past the range, and copes_check reports bit 16."""
    theta = theta_np()
    arena = copes.Arena(canary(N_ALLOC, torch.bfloat16, 9), torch.from_numpy(theta.copy()).cuda())
    sub = make_sub(copes, kind, RANGES, arena)
    big = canary(N_ALLOC, torch.bfloat16, 5)
    before = bits(big).copy()
    short = 20_000  # the range [0, 20000) misses the subspace's upper elements
    copes.perturb_pair(arena, sub, 1, 1e-3, big[:short], 0)
    with pytest.raises(copes.CopesError) as e:
        copes.check()
    assert e.value.code == copes.ERR_DEVICE_CHECK and "bits 0x10" in str(e.value)
    assert np.array_equal(bits(big)[short:], before[short:])
    copes.perturb_partner(arena, sub, big[:short], 0)
    with pytest.raises(copes.CopesError):
        copes.check()
    copes.check()  # cleared


def visit_trace(copes, es, partner_on, kind):
    n = 1 << 18
    theta = theta_np(n, 3)
    arena = copes.Arena(torch.from_numpy(theta.copy()).cuda().to(torch.bfloat16),
                        torch.from_numpy(theta.copy()).cuda())
    layout = copes.Layout([n // 2, n // 2 - 100])
    subs = (es.build_subspaces(layout, "contiguous", 3, tile_size=4096) if kind == "tiles"
            else copes.hash_partition(layout, 3, 5))
    partner = es.Partner.covering(arena, subs) if partner_on else None
    cfg = es.ESConfig(n_members=8, sigma=1e-3, alpha=5e-4)
    rng = np.random.default_rng(1)
    trace = []
    for k, sub in enumerate(subs):
        r = torch.from_numpy(rng.standard_normal(8).astype(np.float32)).cuda()

        def ev(i):  # what a rollout would see: the live weights' bits
            trace.append(int(arena.w.view(torch.int16).to(torch.int64).mul(i + 1).sum()))

        es.round_robin_visit(arena, sub, k, 0, cfg, n, r, evaluate=ev, partner=partner)
    copes.check()
    return trace, bits(arena.w), arena.master.cpu().numpy()


@pytest.mark.parametrize("kind", ["tiles", "indices"])
def test_visit_with_partner_buffer_is_bit_identical(copes, kind):
    from paper_2608_02391_gb300 import es
    t0, w0, m0 = visit_trace(copes, es, False, kind)
    t1, w1, m1 = visit_trace(copes, es, True, kind)
    assert t0 == t1 and len(t0) == 24
    assert np.array_equal(w0, w1)
    assert np.array_equal(m0.view(np.uint32), m1.view(np.uint32))


def test_sync_step_with_partner_buffer_is_bit_identical(copes):
    from paper_2608_02391_gb300 import es
    n, K, N, chunk = 1 << 18, 4, 16, 4096
    layout = copes.Layout([n])
    cfg = es.ESConfig(n_members=N, sigma=1e-3, alpha=5e-4, convention=copes.COEF_PAPER, dimension_aware=True)
    rewards = torch.from_numpy(np.random.default_rng(4).standard_normal(N).astype(np.float32)).cuda()
    out = []
    for use in (False, True):
        theta = theta_np(n, 8)
        arena = copes.Arena(torch.from_numpy(theta.copy()).cuda().to(torch.bfloat16),
                            torch.from_numpy(theta.copy()).cuda())
        subs = es.build_subspaces(layout, "random_chunks", K, seed=9, chunk=chunk)
        partner = es.Partner.covering(arena, subs) if use else None
        for step in range(2):
            es.sync_step(arena, subs, step, cfg, n, rewards, partner=partner)
        out.append((bits(arena.w), arena.master.cpu().numpy().view(np.uint32)))
    copes.check()
    assert np.array_equal(out[0][0], out[1][0]) and np.array_equal(out[0][1], out[1][1])


# ---------------------------------------------------- a second working buffer (w2)
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("kind", ["tiles:1000", "indices", "replay"])
def test_second_buffer_receives_the_context_only(copes, kind, dtype):
    """With copes_params.w2 set, restore, commit, the fused update's commit and init write
    the same values to w2 as to w (on S only); perturbs leave w2 alone."""
    theta = theta_np()
    w_a, w_b = canary(N_ALLOC, dtype, 9), canary(N_ALLOC, dtype, 10)
    dual = copes.Arena(w_a, torch.from_numpy(theta.copy()).cuda(), w2=w_b)
    single = copes.Arena(w_a.clone(), torch.from_numpy(theta.copy()).cuda())
    if kind == "replay":
        layout = copes.Layout([N_ALLOC])
        sub = copes.hash_replay_partition(layout, 3, 11)[1]
        inside = np.zeros(N_ALLOC, bool)
        inside[oracle.hash_list([N_ALLOC], [0], 3, 11, 1).astype(np.int64)] = True
    else:
        sub = make_sub(copes, kind, RANGES, dual)
        inside = mask_of(RANGES)
    b0 = bits(w_b).copy()
    copes.perturb(dual, sub, 5, 1e-3)
    copes.perturb(single, sub, 5, 1e-3)
    assert np.array_equal(bits(dual.w), bits(single.w)) and np.array_equal(bits(w_b), b0)
    copes.restore(dual, sub)
    copes.restore(single, sub)
    got_w, got_w2 = bits(dual.w), bits(w_b)
    assert np.array_equal(got_w, bits(single.w))
    assert np.array_equal(got_w2[inside], got_w[inside]) and np.array_equal(got_w2[~inside], b0[~inside])
    nid, sign, P = copes.member_table(4, copes.ANTITHETIC)
    f = torch.tensor([1.0, -0.5, 0.25, 2.0], device="cuda")
    for a in (dual, single):
        copes.update(a, sub, nid, sign, f, copes.member_seeds(33, 0, 0, P), 0.1, fuse_commit=True)
    assert np.array_equal(dual.master.cpu().numpy().view(np.uint32), single.master.cpu().numpy().view(np.uint32))
    got_w, got_w2 = bits(dual.w), bits(w_b)
    assert np.array_equal(got_w, bits(single.w))
    assert np.array_equal(got_w2[inside], got_w[inside]) and np.array_equal(got_w2[~inside], b0[~inside])
    copes.init_normal(dual, sub, 7, 0.0, 0.02)
    assert np.array_equal(bits(w_b)[inside], bits(dual.w)[inside])
    copes.check()


def dual_trace(copes, es, mode, kind):
    n = 1 << 18
    theta = theta_np(n, 3)
    w = torch.from_numpy(theta.copy()).cuda().to(torch.bfloat16)
    arena = copes.Arena(w, torch.from_numpy(theta.copy()).cuda(), w2=w.clone() if mode == "dual" else None)
    layout = copes.Layout([n // 2, n // 2 - 100])
    subs = (es.build_subspaces(layout, "contiguous", 3, tile_size=4096) if kind == "tiles"
            else copes.hash_replay_partition(layout, 3, 5))
    partner = es.Partner.second_copy(arena) if mode == "dual" else None
    cfg = es.ESConfig(n_members=8, sigma=1e-3, alpha=5e-4)
    rng = np.random.default_rng(1)
    trace = []
    for k, sub in enumerate(subs):
        r = torch.from_numpy(rng.standard_normal(8).astype(np.float32)).cuda()

        def ev(i):  # what a rollout would see: the live buffer's bits
            trace.append(int(arena.live.view(torch.int16).to(torch.int64).mul(i + 1).sum()))

        es.round_robin_visit(arena, sub, k, 0, cfg, n, r, evaluate=ev, partner=partner)
    copes.check()
    return trace, arena


@pytest.mark.parametrize("kind", ["tiles", "replay"])
def test_visit_on_two_working_buffers_is_bit_identical(copes, kind):
    """Members 2j on w and 2j + 1 on w2: every member sees the weights it sees with one
    buffer, and after the visits w, w2 and the master equal the one-buffer run's."""
    from paper_2608_02391_gb300 import es
    t0, a0 = dual_trace(copes, es, "single", kind)
    t1, a1 = dual_trace(copes, es, "dual", kind)
    assert t0 == t1 and len(t0) == 24
    assert np.array_equal(bits(a1.w), bits(a0.w)) and np.array_equal(bits(a1.w2), bits(a0.w))
    assert np.array_equal(a1.master.cpu().numpy().view(np.uint32), a0.master.cpu().numpy().view(np.uint32))


def test_pair_on_an_empty_subspace_is_a_no_op(copes):
    theta = theta_np(1000)
    w = canary(1000, torch.bfloat16, 3)
    arena = copes.Arena(w, torch.from_numpy(theta.copy()).cuda(), w2=w.clone())
    before, before2 = bits(arena.w).copy(), bits(arena.w2).copy()
    empty = copes.tiles_from_ranges([], tile_size=64)
    copes.perturb_pair(arena, empty, 1, 1e-3, arena.w2, 0)
    copes.perturb_partner(arena, empty, arena.w2, 0)
    copes.restore(arena, empty)
    copes.check()
    assert np.array_equal(bits(arena.w), before) and np.array_equal(bits(arena.w2), before2)


# ------------------------------------------- four working copies (w2, w3 and w4)
def quad_arena(copes, theta, dtype):
    cs = [canary(theta.size, dtype, 20 + c) for c in range(4)]
    return copes.Arena(cs[0], torch.from_numpy(theta.copy()).cuda(), *cs[1:])


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("tile", [4096, 1000, 777])
def test_two_pairs_equal_four_perturbs_and_the_oracle(copes, dtype, tile):
    """copes_perturb_two_pairs writes to w, w2, w3 and w4, on S only, exactly what
    copes_perturb writes for (seed_a, +s), (seed_a, -s), (seed_b, +s) and (seed_b, -s),
    and each member agrees with the oracle; ragged and aligned tiles."""
    theta = theta_np()
    inside = mask_of(RANGES)
    g = np.nonzero(inside)[0].astype(np.uint64)
    arena = quad_arena(copes, theta, dtype)
    before = [bits(c).copy() for c in arena.copies]
    ref = copes.Arena(canary(N_ALLOC, dtype, 20), torch.from_numpy(theta.copy()).cuda())
    sub = copes.tiles_from_ranges(RANGES, tile_size=tile)
    for seed_a, seed_b, ss in [(11, 12, 2e-3), (2**40 + 5, 7, -1e-3)]:
        copes.perturb_two_pairs(arena, sub, seed_a, seed_b, ss)
        for c, (seed, s) in enumerate([(seed_a, ss), (seed_a, -ss), (seed_b, ss), (seed_b, -ss)]):
            copes.perturb(ref, sub, seed, s)
            got = bits(arena.copies[c])
            assert np.array_equal(got[inside], bits(ref.w)[inside]), c
            assert np.array_equal(got[~inside], before[c][~inside]), c  # untouched outside S
            check_member(got[inside], dtype, g, theta[inside], seed, s)
    copes.check()


def test_two_pairs_on_an_empty_subspace_is_a_no_op(copes):
    arena = quad_arena(copes, theta_np(1000), torch.bfloat16)
    before = [bits(c).copy() for c in arena.copies]
    copes.perturb_two_pairs(arena, copes.tiles_from_ranges([], tile_size=64), 1, 2, 1e-3)
    copes.check()
    assert all(np.array_equal(bits(c), b) for c, b in zip(arena.copies, before))


@pytest.mark.parametrize("kind", ["tiles:1000", "indices", "replay"])
def test_four_copies_receive_the_context_only(copes, kind):
    """With w2, w3 and w4 set, restore, commit, the fused update's commit and init write
    the same values to every copy as to w (on S only); a plain or pair perturb writes w
    (and the partner buffer) and leaves the other copies alone."""
    theta = theta_np()
    cs = [canary(N_ALLOC, torch.bfloat16, 30 + c) for c in range(4)]
    quad = copes.Arena(cs[0], torch.from_numpy(theta.copy()).cuda(), *cs[1:])
    single = copes.Arena(cs[0].clone(), torch.from_numpy(theta.copy()).cuda())
    if kind == "replay":
        layout = copes.Layout([N_ALLOC])
        sub = copes.hash_replay_partition(layout, 3, 11)[1]
        inside = np.zeros(N_ALLOC, bool)
        inside[oracle.hash_list([N_ALLOC], [0], 3, 11, 1).astype(np.int64)] = True
    else:
        sub = make_sub(copes, kind, RANGES, quad)
        inside = mask_of(RANGES)
    b0 = [bits(c).copy() for c in cs[1:]]

    def others_hold(w_bits):
        for c, b in zip(cs[1:], b0):
            got = bits(c)
            assert np.array_equal(got[inside], w_bits[inside]) and np.array_equal(got[~inside], b[~inside])

    buf = canary(N_ALLOC, torch.bfloat16, 5)
    copes.perturb(quad, sub, 5, 1e-3)
    copes.perturb_pair(quad, sub, 6, 1e-3, buf, 0)
    copes.perturb_pair(single, sub, 6, 1e-3, buf, 0)
    assert np.array_equal(bits(quad.w), bits(single.w))
    assert all(np.array_equal(bits(c), b) for c, b in zip(cs[1:], b0))
    copes.restore(quad, sub)
    copes.restore(single, sub)
    assert np.array_equal(bits(quad.w), bits(single.w))
    others_hold(bits(quad.w))
    nid, sign, P = copes.member_table(4, copes.ANTITHETIC)
    f = torch.tensor([1.0, -0.5, 0.25, 2.0], device="cuda")
    for a in (quad, single):
        copes.update(a, sub, nid, sign, f, copes.member_seeds(33, 0, 0, P), 0.1, fuse_commit=True)
    assert np.array_equal(quad.master.cpu().numpy().view(np.uint32), single.master.cpu().numpy().view(np.uint32))
    assert np.array_equal(bits(quad.w), bits(single.w))
    others_hold(bits(quad.w))
    copes.init_normal(quad, sub, 7, 0.0, 0.02)
    others_hold(bits(quad.w))
    copes.check()


def copies_trace(copes, es, copies, kind, n_members):
    n = 1 << 18
    theta = theta_np(n, 3)
    w = torch.from_numpy(theta.copy()).cuda().to(torch.bfloat16)
    arena = copes.Arena(w, torch.from_numpy(theta.copy()).cuda(), *[w.clone() for _ in range(copies - 1)])
    layout = copes.Layout([n // 2, n // 2 - 100])
    subs = (es.build_subspaces(layout, "contiguous", 3, tile_size=4096) if kind == "tiles"
            else copes.hash_replay_partition(layout, 3, 5))
    partner = {1: None, 2: es.Partner.second_copy, 4: es.Partner.four_copies}[copies]
    partner = partner(arena) if partner else None
    cfg = es.ESConfig(n_members=n_members, sigma=1e-3, alpha=5e-4)
    rng = np.random.default_rng(1)
    trace = []
    for k, sub in enumerate(subs):
        r = torch.from_numpy(rng.standard_normal(n_members).astype(np.float32)).cuda()

        def ev(i):  # what a rollout would see: the live buffer's bits
            trace.append(int(arena.live.view(torch.int16).to(torch.int64).mul(i + 1).sum()))

        es.round_robin_visit(arena, sub, k, 0, cfg, n, r, evaluate=ev, partner=partner)
    copes.check()
    return trace, arena


@pytest.mark.parametrize("kind", ["tiles", "replay"])
@pytest.mark.parametrize("n_members", [8, 6])
def test_visit_on_four_working_copies_is_bit_identical(copes, kind, n_members):
    """Members 4m .. 4m + 3 on w, w2, w3 and w4 (a pair left over goes to w and w2; other
    subspace kinds take pairs): every member sees the weights it sees with one copy, and
    afterwards every copy and the master equal the one-copy run's."""
    from paper_2608_02391_gb300 import es
    t0, a0 = copies_trace(copes, es, 1, kind, n_members)
    t1, a1 = copies_trace(copes, es, 4, kind, n_members)
    assert t0 == t1 and len(t0) == 3 * n_members
    assert all(np.array_equal(bits(c), bits(a0.w)) for c in a1.copies)
    assert np.array_equal(a1.master.cpu().numpy().view(np.uint32), a0.master.cpu().numpy().view(np.uint32))


def test_two_pairs_range_check_reports_without_faulting(copes):
    """A tile past the arena's end: the two-pairs kernel skips it whole, writes no copy
    there, and copes_check reports the device check; the valid tile is written."""
    theta = theta_np(1000)
    arena = quad_arena(copes, theta, torch.bfloat16)
    before = [bits(c).copy() for c in arena.copies]
    bad = copes.SubspaceHandle(copes.SUBSPACE_TILES,
                               torch.tensor([[0, 100], [900, 5000]], dtype=torch.int64, device="cuda"), 0)
    copes.perturb_two_pairs(arena, bad, 1, 2, 1e-3)
    with pytest.raises(copes.CopesError) as e:
        copes.check()
    assert e.value.code == copes.ERR_DEVICE_CHECK
    for c, b in zip(arena.copies, before):
        got = bits(c)
        assert np.array_equal(got[100:], b[100:])  # the bad tile was skipped whole
        assert not np.array_equal(got[:100], b[:100])
    copes.check()  # cleared
