"""Host logic of population-parallel ES on CPU ranks (gloo): the member slices partition
the population, and the reward all-gather returns, on every rank, the full reward vector
bit for bit (including signed zeros, subnormals and infinities a reward could carry)."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rewards(n):
    r = np.random.default_rng(5).standard_normal(n).astype(np.float32)
    special = np.array([-0.0, 1e-45, -3.4e38, np.inf, 0.0], np.float32)
    r[:min(n, special.size)] = special[:min(n, special.size)]
    return r


def _worker(rank, world, port, n, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2608_02391_gb300 import es
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ref = _rewards(n)
        local = np.full(n, np.nan, np.float32)  # other ranks' entries must not leak in
        mine = es.member_slice(rank, world, n)
        local[mine.start:mine.stop] = ref[mine.start:mine.stop]
        got = es.gather_rewards(local, n)
        out.put((rank, got.tobytes(), list(mine)))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,n", [(2, 32), (3, 8), (4, 2)])
def test_reward_all_gather_is_exact_on_every_rank(world, n):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, n, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    ref = _rewards(n).tobytes()
    assert all(r[1] == ref for r in res)
    members = sorted(i for r in res for i in r[2])
    assert members == list(range(n))  # every member evaluated by exactly one rank


def test_member_slices_partition_the_population():
    sys.path.insert(0, ROOT)
    from paper_2608_02391_gb300 import es
    for world in range(1, 9):
        for n in (1, 2, 7, 32, 64, 255):
            got = [i for r in range(world) for i in es.member_slice(r, world, n)]
            assert got == list(range(n))
