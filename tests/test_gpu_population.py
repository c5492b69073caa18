"""Population-parallel ES on the GPU: two ranks (processes) with full replicas of theta
split the members of every visit, exchange the reward scalars over gloo, and apply the
same update (Sec. 3.3: only seeds and scalar rewards travel).  On rank 0 the oracle
recomputes every visit from the gathered rewards -- the shaped fitness, and the update of
Eq. 13 on sampled elements of the subspace (its edges included) -- and the commit is
checked bit for bit.  After a cycle over the K subspaces the ranks' masters and working
weights are bit-identical, and equal to a single process running the whole population.
The ranks' kernels never wait on one another: the only synchronisation is the host
all-gather."""
import datetime
import hashlib
import os
import socket
import sys
import traceback

import numpy as np
import pytest
import torch.multiprocessing as mp

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
N_PARAMS = 1 << 20
K, N = 4, 16


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _setup(copies=1):
    import torch
    sys.path.insert(0, ROOT)
    from paper_2608_02391_gb300 import copes, es
    copes.load()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(0)
    master = torch.empty(N_PARAMS, device="cuda").normal_(0.0, 0.02, generator=gen)
    w = master.to(torch.bfloat16)
    arena = copes.Arena(w, master, *[w.clone() for _ in range(copies - 1)])
    c = torch.empty(N_PARAMS, device="cuda").normal_(0.0, 1.0, generator=gen)
    layout = copes.Layout([N_PARAMS])
    subs = es.build_subspaces(layout, "contiguous", K, tile_size=4096)
    cfg = es.ESConfig(n_members=N, sigma=1e-3, alpha=5e-4, shaping="zscore")
    return torch, copes, es, arena, c, subs, cfg


def _digest(torch, arena):
    """Hash of the master's and the working weights' bits."""
    return hashlib.sha256(arena.master.cpu().numpy().tobytes() +
                          arena.w.view(torch.int16).cpu().numpy().tobytes()).hexdigest()


def _oracle_check(torch, copes, arena, sub, k, cfg, rewards, f_gpu, idx, theta):
    """The visit on subspace k against the oracle at the sampled indices idx (theta: the
    master there before the visit)."""
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import oracle
    from tolerances import assert_fitness_close, assert_update_close
    N = cfg.n_members
    f_ref = oracle.shape_fitness(rewards, oracle.SHAPE_ZSCORE)
    assert_fitness_close(f_gpu, f_ref)
    nid, sign, P = copes.member_table(N, cfg.pairing)
    seeds = copes.member_seeds(cfg.base_seed, 0, k, P)
    coef = np.float32(copes.step_coef(cfg.alpha, N, cfg.sigma, cfg.convention))
    wj = oracle.noise_weights(nid, sign, f_ref, P)
    _, exact, scale = oracle.update_at(idx.astype(np.uint64), theta, seeds, wj, coef)
    it = torch.from_numpy(idx).cuda()
    got = arena.master[it].cpu().numpy()
    assert_update_close(got, exact, scale)
    commit = oracle.bf16_bits_array(got)
    for w in arena.copies:
        assert np.array_equal(w.view(torch.int16)[it].cpu().numpy().view(np.uint16), commit)


def _worker(rank, world, port, out, copies):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    # a bounded collective timeout: a rank that fails ends its peer's next all-gather
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=120))
    try:
        torch, copes, es, arena, c, subs, cfg = _setup(copies)
        # each rank evaluates its antithetic pairs on two working copies, or two pairs at a
        # time on four
        partner = {1: None, 2: es.Partner.second_copy, 4: es.Partner.four_copies}[copies]
        partner = partner(arena) if partner else None

        def evaluate(i):  # the reward of the live perturbation: a linear objective
            return float((c * arena.live.float()).sum().item())

        rng = np.random.default_rng(7)
        width = N_PARAMS // K
        for k in range(K):
            lo, hi = k * width, (k + 1) * width  # subspace k of the contiguous split
            idx = np.unique(np.concatenate([[lo, lo + 1, hi - 2, hi - 1], rng.integers(lo, hi, 3000)]))
            theta = arena.master[torch.from_numpy(idx).cuda()].cpu().numpy()
            rewards = np.zeros(N, np.float32)
            f = es.population_visit(arena, subs[k], k, 0, cfg, N_PARAMS, evaluate, partner=partner,
                                    rewards_out=rewards)
            if rank == 0:
                _oracle_check(torch, copes, arena, subs[k], k, cfg, rewards, f.cpu().numpy(), idx, theta)
        for w in arena.copies[1:]:  # every copy holds the new context
            assert torch.equal(arena.w.view(torch.int16), w.view(torch.int16))
        copes.check()
        digest = _digest(torch, arena)
        ref = None
        if rank == 0:  # the same cycle in one process, whole population
            torch, copes, es, arena1, c1, subs1, cfg1 = _setup()
            for k in range(K):
                rewards = torch.empty(N, device="cuda")

                def ev(i, rewards=rewards):
                    rewards[i] = (c1 * arena1.w.float()).sum()
                es.round_robin_visit(arena1, subs1[k], k, 0, cfg1, N_PARAMS, rewards, evaluate=ev)
            copes.check()
            ref = _digest(torch, arena1)
        out.put((rank, digest, ref, None))
    except Exception:
        out.put((rank, None, None, traceback.format_exc()))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("copies", [1, 2, 4])
def test_two_ranks_match_the_oracle_and_one_process(copies):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out, copies)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted((out.get(timeout=600) for _ in procs), key=lambda t: t[0])
    for p in procs:
        p.join(timeout=120)
    errors = [e for *_, e in res if e]
    assert not errors, "\n".join(errors)
    for p in procs:
        assert p.exitcode == 0
    (r0, d0, ref, _), (r1, d1, _, _) = res
    assert d0 == d1
    assert d0 == ref
