"""Checkpoint / resume: the ES state is the fp32 master plus seeds and the iteration
counter.  A run that is checkpointed to the host after two cycles and resumed in a fresh
arena ends with the same master and weights, bit for bit, as a run that never stopped,
with one working copy, with two (antithetic partners evaluated on the second copy) or with
four (two antithetic pairs at a time)."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

N_PARAMS, K, CYCLES, STOP = 1 << 20, 4, 4, 2


@pytest.fixture(scope="module")
def copes():
    from paper_2608_02391_gb300 import copes as c
    c.load()
    return c


def fresh(copes, copies):
    gen = torch.Generator(device="cuda")
    gen.manual_seed(3)
    master = torch.empty(N_PARAMS, device="cuda").normal_(0.0, 0.02, generator=gen)
    w = master.to(torch.bfloat16)
    return copes.Arena(w, master, *[w.clone() for _ in range(copies - 1)])


def run(copes, es, arena, cfg, cycles, rewards):
    layout = copes.Layout([N_PARAMS])
    subs = es.build_subspaces(layout, "contiguous", K, tile_size=4096)
    partner = {1: None, 2: es.Partner.second_copy, 4: es.Partner.four_copies}[len(arena.copies)]
    partner = partner(arena) if partner else None
    for t in cycles:
        for k in range(K):
            r = torch.from_numpy(rewards[t * K + k]).cuda()
            es.round_robin_visit(arena, subs[k], k, t, cfg, N_PARAMS, r, partner=partner)


@pytest.mark.parametrize("copies", [1, 2, 4], ids=["one-copy", "two-copies", "four-copies"])
def test_resume_is_bit_exact(copes, tmp_path, copies):
    from paper_2608_02391_gb300 import es
    cfg = es.ESConfig(n_members=16, sigma=1e-3, alpha=5e-4, shaping="centered_rank")
    rewards = np.random.default_rng(4).integers(0, 9, (CYCLES * K, 16)).astype(np.float32) / 8
    straight = fresh(copes, copies)
    run(copes, es, straight, cfg, range(CYCLES), rewards)
    first = fresh(copes, copies)
    run(copes, es, first, cfg, range(STOP), rewards)
    path = tmp_path / "state.pt"
    torch.save(es.state_dict(first, cfg, STOP), path)
    del first
    resumed, cfg2, t0 = es.load_state(torch.load(path))
    assert t0 == STOP and cfg2 == cfg
    assert len(resumed.copies) == copies
    run(copes, es, resumed, cfg2, range(t0, CYCLES), rewards)
    copes.check()
    assert torch.equal(resumed.master.view(torch.int32), straight.master.view(torch.int32))
    assert torch.equal(resumed.w.view(torch.int16), straight.w.view(torch.int16))
    for mine, theirs in zip(resumed.copies[1:], straight.copies[1:]):
        assert torch.equal(mine.view(torch.int16), theirs.view(torch.int16))
        assert torch.equal(mine.view(torch.int16), resumed.w.view(torch.int16))
