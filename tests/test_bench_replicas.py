"""The benchmark's multi-rank logic on CPU ranks (gloo, world size 2): every rank runs an
independent replica, the slowest rank's time counts, and the job throughput is the sum of
the replicas' work over that time. Only rank 0 prints the reference line."""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 100.0 + 50.0 * rank  # rank 1 is the slow one
        ms = bench.max_over_ranks(local_ms)
        out.put((rank, ms, bench.job_throughput(world, 1000, 5, ms * 1e-3)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_throughput_gloo():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [150.0, 150.0]  # both ranks see the slowest time
    assert res[0][2] == pytest.approx(2 * 1000 * 5 / 0.150)


def test_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(1, 10, 2, 4.0) == 5.0


def test_reference_arm_prints_only_on_rank_0():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0", "--cpu-sample", "4096"],
                         capture_output=True, text=True, env=env, timeout=300)
    assert res.returncode == 0 and res.stdout.strip() == ""
    env = dict(os.environ, RANK="0", WORLD_SIZE="1", LOCAL_RANK="0")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "1", "--warmup", "0", "--cpu-sample", "4096"],
                         capture_output=True, text=True, env=env, timeout=300)
    assert res.returncode == 0
    import json
    line = json.loads(res.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "params/s" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["e2e"]["h2d_bytes_per_step"] == 0


def test_clock_sampler_names_the_physical_gpu(monkeypatch):
    """nvidia-smi ignores CUDA_VISIBLE_DEVICES: without a CUDA device to give its UUID,
    the local index is mapped through the visible-device list."""
    sys.path.insert(0, ROOT)
    import bench
    import torch
    if torch.cuda.is_available():
        uuid = bench.smi_gpu_id(0)
        assert uuid.startswith(("GPU-", "MIG-"))
        return
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "5,GPU-1234")
    assert bench.smi_gpu_id(0) == "5" and bench.smi_gpu_id(1) == "GPU-1234"
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "")
    assert bench.smi_gpu_id(3) == "3"
