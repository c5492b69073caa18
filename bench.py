#!/usr/bin/env python
"""ES-iteration throughput of the CoPES core on GB300.

Workload: 4B-parameter decoder-shaped set (36 layers, hidden 2560, MLP 9728, vocab 151936,
tied embeddings; 4,022,468,096 parameters), bf16 working weights + fp32 master (24 GB
resident, plus three more 8 GB working copies by default), K = 8 layer-block subspaces,
N = 32 antithetic members, sigma = 1e-3, alpha = 5e-4, z-score shaping, step coefficient
alpha / (N sigma).

One step = one cooperative-coevolution cycle: for each of the 8 subspaces, rebuild its
tile table (the partition step), perturb the 32 members (rewards are seeded synthetic
scalars, no model is evaluated), restore, fitness shaping and the fused update + context
commit.  Every parameter passes through 32 member perturbations, one restore and one
update per step, so value = parameters per step x steps / time.  `--weights` picks how
the members are materialised: `quad` (default) writes antithetic members 4m .. 4m+3 (two
noise vectors) to four working copies in one pass; `dual` writes members 2j and 2j+1 to
two copies in one pass; `partner` keeps one copy and copies member 2j+1 in from a partner
buffer; `single` perturbs every member from theta.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl copes|reference]

`--case 4b-sync` times the paper's Algorithm 1 step on the 4B set: a random equal-size
chunk partition (K = 4, chunks of 65,536) resampled every step, N = 32 antithetic members
split N_k = 8 per subspace, dimension-aware sigma_k, joint z-score and the composed
update with coefficient alpha / N_k.

`--case 4b-backup` times the 4B step in the CPU weight backup mode: bf16 weights on the
GPU, the context in pinned host memory, no fp32 master.

`--case 4b-hash` times the non-contiguous workload instead: the same 4B set split by a
per-element hash into K = 16 subspaces, N = 64 antithetic members, one step = one sweep
over the 16 subspaces, with the subspaces replayed from the partition seed (default;
`--hash-mode replay-mask` hashes once per visit into a membership mask) or
read from int64 index lists (`--hash-mode lists`), or read from index lists with each
subspace's theta kept in list order (`--hash-mode gathered`).

Prints one JSON line (rank 0).  Under torchrun each rank runs an independent replica on
its own GPU (the path needs no exchange at this scope), timed with a barrier and the max
over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ES-iteration params/s and HBM GB/s at 4B bf16 (N=32), % of roofline on 1 GB300"
FALLBACK_HBM_GBS = 6800.0

# ncu DRAM bytes per element of the dominant kernel (the two-pairs perturb, the pair
# perturb under --weights dual or partner, the plain perturb under --weights single; bf16)
# from one capture each; a figure is dropped (traffic = null) when the tile kernels'
# sources (source_sha) no longer match the hash it was taken on.  The figures come from
# subspaces of 2^28 parameters, where the writes still in L2 when the kernel ends are about
# 2% of its traffic.
NCU_TRAFFIC = {
    "perturb_two_pairs": {"kernel": "elem_tiles_kernel<perturb_two_pairs,bf16>", "source_sha": "2d16bf01a43641d5",
                          "bytes_per_elem": 11.782, "capture": "profiles/perturb_two_pairs_4b_slice.md",
                          "case": "two 2^28-parameter subspaces (--case 4b-slice-big)"},
    "perturb_pair": {"kernel": "elem_tiles_kernel<perturb_pair,bf16>", "source_sha": "2d16bf01a43641d5",
                     "bytes_per_elem": 7.827, "capture": "profiles/perturb_pair_4b_slice.md",
                     "case": "two 2^28-parameter subspaces (--case 4b-slice-big --weights dual)"},
    "perturb": {"kernel": "elem_tiles_kernel<perturb,bf16>", "source_sha": "2d16bf01a43641d5",
                "bytes_per_elem": 5.862, "capture": "profiles/perturb_4b_slice.md",
                "case": "two 2^28-parameter subspaces (--case 4b-slice-big --weights single)"},
}


WEIGHTS_MODES = {
    "quad": "four bf16 copies: antithetic members 4m, 4m+1 (noise 2m) and 4m+2, 4m+3 (noise 2m+1) evaluated "
            "on w, w2, w3, w4, all four written by one two-pairs perturb",
    "dual": "two bf16 copies: antithetic member 2j evaluated on w, 2j+1 on w2, both written by one pair perturb",
    "partner": "one bf16 copy: member 2j+1 copied in from the pair perturb's partner buffer",
    "single": "one bf16 copy: every member perturbed from theta",
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="copes", choices=["copes", "reference"])
    ap.add_argument("--tile", type=int, default=1 << 14)
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--cpu-sample", type=int, default=1 << 20,
                    help="parameters of the oracle's timed CPU sample")
    ap.add_argument("--weights", default=None, choices=["quad", "dual", "partner", "single"],
                    help="quad (default for the round-robin tile cases): four working-weight copies, two "
                         "antithetic pairs written by one pass; dual (default for the hash, backup and sync "
                         "cases): two "
                         "working-weight copies, antithetic members 2j on w and 2j+1 on w2 (one pair "
                         "perturb per pair; the backup case keeps one copy and a partner buffer); partner: "
                         "one copy, member 2j+1 copied in from a partner buffer; single: one copy, every "
                         "member perturbed from theta")
    ap.add_argument("--cpu-cores", type=int, default=0,
                    help="processes of the oracle's CPU sample (0: every core this process may use)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-kernels", type=int, default=1,
                    help="1: add the oracle's single-thread per-kernel timings (tiny workload and a "
                         "0.5B subspace sample) to cpu_baseline; 0: skip them")
    ap.add_argument("--case", default="4b", choices=["4b", "0.5b", "8b", "4b-slice", "4b-slice-big", "4b-hash",
                                                     "4b-hash-slice", "4b-backup", "4b-backup-slice", "4b-sync"],
                    help="4b: the benchmark workload; 0.5b: the 0.5B set (K=8 layer groups, N=16, centred "
                         "rank); 8b: the 8B set (K=4 type groups, N=128, sigma 5e-4; one step = one of its "
                         "10 CC cycles); 4b-slice: a 268M-parameter case for profiling; 4b-slice-big: two "
                         "2^28-parameter subspaces, for DRAM-traffic captures; "
                         "4b-hash: one sweep over the 16 hash subspaces of the 4B set (N=64); "
                         "4b-hash-slice: the same on 268M parameters, for profiling; "
                         "4b-backup: the 4B step in the CPU weight backup mode (no fp32 master); "
                         "4b-backup-slice: the same on 268M parameters, for profiling; "
                         "4b-sync: Algorithm 1 on the 4B set (K=4 random chunks resampled each step)")
    ap.add_argument("--hash-mode", default="replay", choices=["replay", "replay-mask", "lists", "gathered"],
                    help="4b-hash: subspaces replayed from the partition seed (hashing in every kernel, "
                         "or once per visit into a membership mask), int64 index lists, or index lists "
                         "with a gathered (list-order) master per subspace")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value: float, device="cpu") -> float:
    """The largest of every rank's value (identity when not distributed)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, units_per_step: int, steps: int, seconds: float) -> float:
    """Whole-job throughput of N independent replicas: every rank processes the full
    workload, the slowest rank's time counts (weak scaling)."""
    return world * units_per_step * steps / seconds


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            return json.load(fh), "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


def source_sha():
    """Hash of the code the tile kernels compile from: comments and blank space are
    dropped first, so an edit to a comment keeps a capture valid and any code change
    drops it."""
    h = hashlib.sha256()
    for name in ("es_kernels.cu", "copes_device.cuh", "copes_internal.h", "es_common.cuh", "normal_coeffs.h"):
        with open(os.path.join(ROOT, "paper_2608_02391_gb300", "csrc", name)) as fh:
            text = re.sub(r"/\*.*?\*/", "", fh.read(), flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        h.update("\n".join(line.strip() for line in text.splitlines() if line.strip()).encode())
    return h.hexdigest()[:16]


def smi_gpu_id(local: int) -> str:
    """The nvidia-smi identifier of torch device `local`.  nvidia-smi numbers GPUs
    physically and ignores CUDA_VISIBLE_DEVICES, so the device is named by its UUID;
    failing that, CUDA_VISIBLE_DEVICES maps the local index to the physical one."""
    try:
        import torch
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        if uuid:
            return uuid if uuid.startswith(("GPU-", "MIG-")) else "GPU-" + uuid
    except Exception:
        pass
    visible = [v.strip() for v in os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",") if v.strip()]
    return visible[local] if local < len(visible) else str(local)


class ClockSampler:
    """nvidia-smi clocks / throttle reasons of one GPU, sampled every 200 ms while running."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local: int):
        self.gpu = smi_gpu_id(local)
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu, f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "gpu": self.gpu}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "gpu": self.gpu}


# ------------------------------------------------------------------------ CPU oracle leg
def oracle_visit_sample(wl, n_sample: int, iteration: int = 0, part: int = 0):
    """The oracle as it stands on a bounded sample: one subspace visit (N perturbs,
    restore, shaping, fused update + commit) restricted to parameters
    [part * n_sample, (part + 1) * n_sample) of subspace 0.  Returns (seconds, parameters)."""
    import oracle
    from paper_2608_02391_gb300 import workloads
    N = wl.n_members
    b = part * n_sample
    rng = np.random.default_rng(part)
    master = np.zeros(b + n_sample, np.float32)  # pages below b are never touched
    master[b:] = rng.standard_normal(n_sample) * 0.02
    w = np.zeros(b + n_sample, np.uint16)
    sub = oracle.make_subspace(ranges=[(b, b + n_sample)])
    nid, sign, P = oracle.member_table(N, oracle.ANTITHETIC)
    seeds = np.array([oracle.member_seed(wl.base_seed, iteration, 0, j) for j in range(P)], np.uint64)
    rewards = workloads.reward_stream(wl, 1)[0]
    t0 = time.perf_counter()
    for i in range(N):
        oracle.perturb(w, master, sub, int(seeds[nid[i]]), float(sign[i]) * wl.sigma)
    oracle.restore(w, master, sub)
    f = oracle.shape_fitness(rewards, oracle_shaping(wl))
    coef = np.float32(oracle.step_coef(wl.alpha, N, wl.sigma, oracle.COEF_OPENAI))
    oracle.update(master, sub, nid, sign, f, seeds, coef, w=w)
    return time.perf_counter() - t0, n_sample


def oracle_shaping(wl):
    import oracle
    return {"zscore": oracle.SHAPE_ZSCORE, "zscore_grouped": oracle.SHAPE_ZSCORE_GROUPED,
            "centered_rank": oracle.SHAPE_CENTERED_RANK, "none": oracle.SHAPE_NONE}[wl.shaping]


def oracle_kernel_timings(wl, n_sample: int) -> dict:
    """The oracle's kernels one at a time on one host thread, over n_sample parameters
    of a subspace of workload wl (bf16 working weights, its N, sigma and shaping): mean
    time per call of perturb (two members), restore, shaping and the update with its
    fused commit, as parameters/s and algorithmic GB/s (the GPU kernels' units)."""
    import oracle
    from paper_2608_02391_gb300 import workloads
    N = wl.n_members
    rng = np.random.default_rng(1)
    master = (rng.standard_normal(n_sample) * 0.02).astype(np.float32)
    w = np.zeros(n_sample, np.uint16)
    sub = oracle.make_subspace(ranges=[(0, n_sample)])
    nid, sign, P = oracle.member_table(N, oracle.ANTITHETIC)
    seeds = np.array([oracle.member_seed(wl.base_seed, 0, 1, j) for j in range(P)], np.uint64)
    rewards = workloads.reward_stream(wl, 1)[0]

    def timed(fn, reps=1):
        t0 = time.perf_counter()
        for r in range(reps):
            fn(r)
        return (time.perf_counter() - t0) / reps

    t_perturb = timed(lambda r: oracle.perturb(w, master, sub, int(seeds[nid[r]]), float(sign[r]) * wl.sigma), 2)
    t_restore = timed(lambda r: oracle.restore(w, master, sub))
    f = oracle.shape_fitness(rewards, oracle_shaping(wl))
    t_shape = timed(lambda r: oracle.shape_fitness(rewards, oracle_shaping(wl)), 100)
    coef = np.float32(oracle.step_coef(wl.alpha, N, wl.sigma, oracle.COEF_OPENAI))
    t_update = timed(lambda r: oracle.update(master, sub, nid, sign, f, seeds, coef, w=w))
    per = lambda t, b: {"ms": 1e3 * t, "params/s": n_sample / t, "GB/s": b * n_sample / t / 1e9}
    return {"perturb": per(t_perturb, 6.0), "restore": per(t_restore, 6.0),
            "shape": {"ms": 1e3 * t_shape, "members": N},
            "update_fused_commit": {**per(t_update, 10.0), "normals_per_elem": P}}


def host_cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                name = line.split(":", 1)[1].strip()
                if name and not name.isdigit():
                    return name
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as fh:
            for line in fh:
                if line.lower().startswith(("model name", "hardware")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


def _oracle_part(args):
    return oracle_visit_sample(*args)


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


class OraclePool:
    """The oracle on every host core: one spawned process per core (spawn, not fork: the
    parent may hold a CUDA context), each running the same visit on its own disjoint
    range of subspace 0.  Throughput = all ranges' parameters / the wall time of the
    parallel map."""

    def __init__(self, wl, cores: int):
        import multiprocessing as mp
        import oracle
        oracle.build()
        self.wl, self.cores = wl, max(1, cores)
        self.pool = mp.get_context("spawn").Pool(self.cores) if self.cores > 1 else None

    def visit(self, n_per_core: int, iteration: int = 0):
        jobs = [(self.wl, n_per_core, iteration, part) for part in range(self.cores)]
        t0 = time.perf_counter()
        res = self.pool.map(_oracle_part, jobs, chunksize=1) if self.pool else [_oracle_part(jobs[0])]
        wall = time.perf_counter() - t0
        return wall, sum(m for _, m in res)

    def close(self):
        if self.pool:
            self.pool.close()
            self.pool.join()


def run_reference(args, wl):
    rank, world, _ = dist_env()
    if world > 1 and rank != 0:
        return
    n = max(1024, args.cpu_sample // 4)
    pool = OraclePool(wl, args.cpu_cores or host_cores())
    try:
        pool.visit(1024)  # loads the oracle in every worker
        for _ in range(max(args.warmup, 0)):
            pool.visit(1024)
        tot_t, tot_n = 0.0, 0
        for s in range(args.steps):
            t, m = pool.visit(n, iteration=s)
            tot_t += t
            tot_n += m
    finally:
        pool.close()
    value = tot_n / tot_t
    sample = (f"each step: one subspace visit (N={wl.n_members} perturbs, restore, {wl.shaping} shaping, "
              f"fused update + commit) over {n} parameters per core, {pool.cores} processes on "
              f"disjoint ranges of subspace 0")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(wl, args),
        "cpu_baseline": {"value": value, "unit": "params/s", "cores": pool.cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "params/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


DECODER_SETS = {
    "4b": ("4B decoder-shaped bf16 set, fp32 master, K=8 layer blocks, N=32 antithetic",
           {"layers": 36, "hidden": 2560, "mlp": 9728, "vocab": 151936, "tied": True},
           "24 GB or more resident per step"),
    "0.5b": ("0.5B decoder-shaped bf16 set, fp32 master, K=8 layer groups (embeddings alone), N=16 antithetic",
             {"layers": 24, "hidden": 896, "mlp": 4864, "vocab": 151936, "tied": True},
             "3 GB or more resident per step"),
    "8b": ("8B decoder-shaped bf16 set, fp32 master, K=4 subspaces by parameter type, N=128 antithetic; "
           "one step = one cycle of the 10-cycle CC loop",
           {"layers": 36, "hidden": 4096, "mlp": 12288, "vocab": 151936, "tied": False},
           "49 GB or more resident per step"),
}


def workload_config(wl, args):
    if wl.name not in DECODER_SETS:
        return {"workload": f"{wl.name}: {wl.d} parameters in {len(wl.tensors)} tensors, K={wl.K}, "
                            f"N={wl.n_members} antithetic (profiling case)", "params": wl.d, "K": wl.K,
                "N": wl.n_members, "tile": args.tile}
    desc, shape, resident = DECODER_SETS[wl.name]
    return {"workload": desc, "params": wl.d, **shape,
            "K": wl.K, "N": wl.n_members, "sigma": wl.sigma, "alpha": wl.alpha, "shaping": wl.shaping,
            "tile": args.tile, "working_weights": WEIGHTS_MODES[args.weights],
            "l2": f"inputs larger than L2 ({resident}), no flush"}


# -------------------------------------------------------------------------- GPU leg
def n_copies(args) -> int:
    """Working-weight copies of --weights."""
    return {"quad": 4, "dual": 2}.get(args.weights, 1)


def perturb_kernel(args) -> str:
    """The member perturb --weights times (an N that is a multiple of 4 under quad)."""
    return {"quad": "perturb_two_pairs", "single": "perturb"}.get(args.weights, "perturb_pair")


def make_arena(copes, torch, wl, layout, copies=1):
    """Seeded synthetic weights: fp32 master ~ N(0, init_scale^2), norm tensors 1.0, and
    w = bf16(master) (and the further working copies = w)."""
    master = torch.empty(layout.d_pad, dtype=torch.float32, device="cuda")
    gen = torch.Generator(device="cuda")
    gen.manual_seed(wl.init_seed)
    master.normal_(0.0, wl.init_scale, generator=gen)
    offs = layout.offsets
    for t, ten in enumerate(wl.tensors):
        if ten.kind == "norm":
            master[int(offs[t]):int(offs[t]) + ten.numel].fill_(1.0)
    w = master.to(torch.bfloat16)
    return copes.Arena(w, master, *[w.clone() for _ in range(copies - 1)])


def main():
    args = parse()
    from paper_2608_02391_gb300 import workloads
    wl = workloads.workload({"4b-backup": "4b", "4b-sync": "4b", "4b-backup-slice": "4b-slice"}.get(args.case, args.case))
    if args.weights is None:  # four copies pay off where a restore serves many members
        args.weights = "quad" if wl.mode != "hash" and args.case not in ("4b-backup", "4b-backup-slice",
                                                                          "4b-sync") else "dual"
    if args.impl == "reference":
        return run_reference(args, wl)

    import torch
    from paper_2608_02391_gb300 import copes, es
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    copes.load()
    if args.weights == "quad" and (wl.mode == "hash" or args.case in ("4b-backup", "4b-backup-slice")):
        raise SystemExit("--weights quad needs tile subspaces and an fp32 master: not for --case " + args.case)
    if wl.mode == "hash":
        return run_hash(args, wl, copes, es, torch, rank, world, local)
    if args.case in ("4b-backup", "4b-backup-slice"):
        return run_backup(args, wl, copes, es, torch, rank, world, local)
    if args.case == "4b-sync":
        return run_sync(args, wl, copes, es, torch, rank, world, local)

    layout = copes.Layout(wl.numel)
    d = wl.d
    arena = make_arena(copes, torch, wl, layout, copies=n_copies(args))
    cfg = es.ESConfig(n_members=wl.n_members, sigma=wl.sigma, alpha=wl.alpha, shaping=wl.shaping)
    total_steps = args.warmup + args.steps + args.e2e_steps
    rewards_host = workloads.reward_stream(wl, total_steps * wl.K)  # [steps*K, N]
    rewards_dev = torch.from_numpy(rewards_host).cuda()
    fitness = torch.empty(wl.n_members, dtype=torch.float32, device="cuda")
    spec_groups = np.ascontiguousarray(wl.group_of, np.int32)
    subs = es.build_subspaces(layout, "groups", wl.K, group_of=wl.group_of, tile_size=args.tile)
    tile_buf = [s.tensor for s in subs]
    # antithetic pairs: one noise generation per pair, the partner's weights staged in a
    # buffer as wide as the widest subspace
    if args.weights == "quad":
        partners = [es.Partner.four_copies(arena)] * wl.K
    elif args.weights == "dual":
        partners = [es.Partner.second_copy(arena)] * wl.K
    elif args.weights == "partner":
        partners = es.Partner.per_subspace(arena, subs)
    else:
        partners = [None] * wl.K

    import ctypes
    L = copes.load()

    def rebuild(k):
        """The partition step for subspace k: recompute its tile table into its buffer."""
        spec = copes.PartitionSpec(copes.PART_TENSOR_GROUPS, wl.K, 0, 0,
                                   spec_groups.ctypes.data_as(ctypes.c_void_p))
        cnt = ctypes.c_uint64()
        copes._check(L.copes_subspace_build(ctypes.byref(layout.desc), ctypes.byref(spec), k, args.tile, None,
                                            ctypes.c_void_p(tile_buf[k].data_ptr()), tile_buf[k].shape[0],
                                            ctypes.byref(cnt), copes._stream(None)))

    def step(s, events=None):
        for k in range(wl.K):
            es._timed(events, "rebuild", lambda: rebuild(k))  # one tile-expansion kernel
            es.round_robin_visit(arena, subs[k], k, s, cfg, d, rewards_dev[s * wl.K + k],
                                 fitness_out=fitness, events=events, partner=partners[k])

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    copes.check()
    if world > 1:
        dist.barrier()

    events = {}
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        start.record()
        for s in range(args.warmup, args.warmup + args.steps):
            step(s, events)
        end.record()
        torch.cuda.synchronize()
    ms = max_over_ranks(start.elapsed_time(end), "cuda")
    copes.check()

    # end to end through the public API: rewards from pinned host memory each visit,
    # the shaped fitness read back each step, host wall clock
    pinned = torch.from_numpy(rewards_host).pin_memory()
    fit_host = torch.empty((wl.K, wl.n_members), dtype=torch.float32).pin_memory()
    r_dev = torch.empty(wl.n_members, dtype=torch.float32, device="cuda")
    f_all = torch.empty((wl.K, wl.n_members), dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    s0 = args.warmup + args.steps
    e2e_events = {}  # the same per-kernel event records as the timed region
    for s in range(s0, s0 + args.e2e_steps):
        for k in range(wl.K):
            rebuild(k)
            r_dev.copy_(pinned[s * wl.K + k], non_blocking=True)
            es.round_robin_visit(arena, subs[k], k, s, cfg, d, r_dev, fitness_out=f_all[k],
                                 events=e2e_events, partner=partners[k])
        fit_host.copy_(f_all, non_blocking=True)
        torch.cuda.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, "cuda")

    if rank != 0:
        dist.destroy_process_group() if world > 1 else None
        return

    # per-kernel average launch times (CUDA events on the launching stream)
    per = {name: float(np.mean([a.elapsed_time(b) for a, b in lst])) for name, lst in events.items()}
    counts = {name: len(lst) for name, lst in events.items()}
    d_k = [s.numel for s in subs]
    mean_dk = float(np.mean(d_k))
    peaks, peak_src = measured_peaks()
    hbm = float(peaks["hbm_gbs"])
    copies = n_copies(args)
    pk = perturb_kernel(args)
    # the pair perturb reads theta (4 B) and writes w and the partner's weights (2 + 2 B);
    # the two-pairs perturb reads theta and writes four copies (4 + 4 x 2 B); the partner
    # copy reads and writes 2 B; a plain perturb reads 4 B and writes 2 B.  Restore and
    # the fused commit write every working copy (2 B each).
    perturb_bytes = {"perturb_two_pairs": 12.0, "perturb_pair": 8.0, "perturb": 6.0}[pk] * mean_dk
    restore_bytes = (4.0 + 2.0 * copies) * mean_dk
    update_bytes = (8.0 + 2.0 * copies) * mean_dk
    achieved = perturb_bytes / (per["perturb"] * 1e-3) / 1e9
    ncu = NCU_TRAFFIC.get(pk, {"source_sha": None})
    traffic = None
    if ncu["source_sha"] == source_sha() and ncu["bytes_per_elem"]:
        traffic = ncu["bytes_per_elem"] * mean_dk
        traffic_note = (f"ncu dram__bytes_read + dram__bytes_write per element ({ncu['bytes_per_elem']} B) "
                        f"on {ncu.get('case', 'a 2^26-parameter subspace')}, times this launch's elements")
    else:
        traffic_note = "no capture for the current kernel sources"
    props = torch.cuda.get_device_properties(local)
    clk = clocks.summary()
    n_normals_update = wl.n_members // 2
    alu_ops_per_normal = 28  # pinned algorithmic op count: 27 per normal + 1 fma
    sm_mhz = clk["sm_mhz"] or float(peaks.get("sm_max_mhz", 2070.0))
    alu_peak = props.multi_processor_count * 128 * sm_mhz * 1e6 / 1e12  # Tops/s at the sampled clock
    upd_ops = mean_dk * n_normals_update * alu_ops_per_normal / (per["update"] * 1e-3) / 1e12
    members_bytes = {"perturb_two_pairs": (wl.n_members // 4) * 12, "perturb_pair": (wl.n_members // 2) * 8,
                     "perturb": wl.n_members * 6}[pk] + (wl.n_members // 2) * 4 * (args.weights == "partner")
    bytes_per_step = d * (members_bytes + (4 + 2 * copies) + (8 + 2 * copies))
    value = job_throughput(world, d, args.steps, ms * 1e-3)
    e2e = job_throughput(world, d, args.e2e_steps, e2e_s)
    launches = sum(counts.values())
    out = {
        "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_config(wl, args),
        "hbm_gbs": bytes_per_step * args.steps / (ms * 1e-3) / 1e9,
        "roofline": {"bound": "hbm", "kernel": pk, "achieved": achieved,
                     "peak": hbm, "unit": "GB/s", "frac": achieved / hbm, "traffic": traffic,
                     "traffic_source": traffic_note,
                     "peak_source": peak_src, "algorithmic_bytes_per_launch": perturb_bytes},
        "kernels": {
            pk: {"ms": per["perturb"], "launches": counts["perturb"], "GB/s": achieved, "frac_hbm": achieved / hbm,
                 # pinned lane-ops: 27 per normal, 3 per member written (fma, round, pack)
                 **({"frac_alu": (2 * 27 + 4 * 3) * mean_dk / (per["perturb"] * 1e-3) / (alu_peak * 1e12),
                     "ops_per_elem": 2 * 27 + 4 * 3} if pk == "perturb_two_pairs" else {})},
            "restore": {"ms": per["restore"], "launches": counts["restore"],
                        "GB/s": restore_bytes / (per["restore"] * 1e-3) / 1e9,
                        "frac_hbm": restore_bytes / (per["restore"] * 1e-3) / 1e9 / hbm},
            "update_fused_commit": {"ms": per["update"], "launches": counts["update"],
                                    "GB/s": update_bytes / (per["update"] * 1e-3) / 1e9,
                                    "bound": "alu", "achieved_Tops": upd_ops, "peak_Tops": alu_peak,
                                    "frac_alu": upd_ops / alu_peak,
                                    "ops_per_normal": alu_ops_per_normal, "normals_per_elem": n_normals_update},
            "shape": {"ms": per["shape"], "launches": counts["shape"]},
            "tile_rebuild": {"ms": per["rebuild"], "launches": counts["rebuild"]},
            **({"perturb_partner": {"ms": per["partner"], "launches": counts["partner"],
                                    "GB/s": 4.0 * mean_dk / (per["partner"] * 1e-3) / 1e9,
                                    "frac_hbm": 4.0 * mean_dk / (per["partner"] * 1e-3) / 1e9 / hbm}}
               if "partner" in per else {}),
        },
        "clocks": clk,
        "e2e": {"value": e2e, "unit": "params/s", "h2d_bytes_per_step": wl.K * wl.n_members * 4,
                "d2h_bytes_per_step": wl.K * wl.n_members * 4},
        "gpu_launches": launches,
    }
    if not args.no_cpu_baseline and world == 1:
        pool = OraclePool(wl, args.cpu_cores or host_cores())
        try:
            pool.visit(1024)  # loads the oracle in every worker
            t, m = pool.visit(args.cpu_sample)
        finally:
            pool.close()
        out["cpu_baseline"] = {
            "value": m / t, "unit": "params/s", "cores": pool.cores, "kind": "oracle",
            "cpu_model": host_cpu_model(),
            "sample": f"one subspace visit (N={wl.n_members} perturbs, restore, shaping, fused update + "
                      f"commit) over {args.cpu_sample} parameters per core, {pool.cores} processes on "
                      f"disjoint ranges of subspace 0 ({m} parameters), {t:.1f} s"}
        if args.cpu_kernels:
            from paper_2608_02391_gb300 import workloads
            n_k = 1 << 20
            out["cpu_baseline"]["single_thread_kernels"] = {
                "tiny": {"sample": f"{n_k} parameters, the tiny workload's N=8 and z-score, bf16 working "
                                   "weights", **oracle_kernel_timings(workloads.workload("tiny"), n_k)},
                "0.5b": {"sample": f"{n_k} parameters of a 0.5B subspace, N=16, centred rank, bf16 working "
                                   "weights", **oracle_kernel_timings(workloads.workload("0.5b"), n_k)}}
    print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_hash(args, wl, copes, es, torch, rank, world, local):
    """The 4B-hash sweep: each of the K = 16 hash subspaces gets one ES iteration with
    N = 64 members (perturbs, restore, shaping, fused update + commit)."""
    from paper_2608_02391_gb300 import workloads
    layout = copes.Layout(wl.numel, list(range(len(wl.tensors))))
    d = wl.d
    arena = make_arena(copes, torch, wl, layout, copies=n_copies(args))
    # a hash subspace spreads over the whole arena: the partner is w2 or a full-size buffer
    if args.weights == "dual":
        partner = es.Partner.second_copy(arena)
    elif args.weights == "partner":
        partner = es.Partner(torch.empty(layout.d_pad, dtype=arena.w.dtype, device="cuda"), 0)
    else:
        partner = None
    mask_buf = None
    if args.hash_mode in ("replay", "replay-mask"):
        subs = copes.hash_replay_partition(layout, wl.K, wl.partition_seed)
        if args.hash_mode == "replay-mask":  # one mask buffer, rebuilt at every visit
            mask_buf = torch.empty(int(subs[0].replay.n_replay_tiles) * 512, dtype=torch.int32, device="cuda")
    else:
        subs = copes.hash_partition(layout, wl.K, wl.partition_seed)
        if args.hash_mode == "gathered":  # each subspace's theta in list order (contiguous reads)
            for sub in subs:
                copes.gather_master(arena, sub)
    cfg = es.ESConfig(n_members=wl.n_members, sigma=wl.sigma, alpha=wl.alpha, shaping=wl.shaping)
    total_steps = args.warmup + args.steps
    rewards = torch.from_numpy(workloads.reward_stream(wl, total_steps * wl.K)).cuda()
    fitness = torch.empty(wl.n_members, dtype=torch.float32, device="cuda")

    def step(s, events=None):
        for k in range(wl.K):
            if mask_buf is not None:
                es._timed(events, "mask", lambda: copes.hash_replay_mask(arena, subs[k], mask_buf))
            es.round_robin_visit(arena, subs[k], k, s, cfg, d, rewards[s * wl.K + k], fitness_out=fitness,
                                 events=events, partner=partner)

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    copes.check()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    events = {}
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        start.record()
        for s in range(args.warmup, args.warmup + args.steps):
            step(s, events)
        end.record()
        torch.cuda.synchronize()
    ms = max_over_ranks(start.elapsed_time(end), "cuda")
    copes.check()
    if rank != 0:
        return
    per = {name: float(np.mean([a.elapsed_time(b) for a, b in lst])) for name, lst in events.items()}
    counts = {name: len(lst) for name, lst in events.items()}
    mean_dk = float(np.mean([s.numel for s in subs]))
    peaks, peak_src = measured_peaks()
    hbm = float(peaks["hbm_gbs"])
    props = torch.cuda.get_device_properties(local)
    clk = clocks.summary()
    sm_mhz = clk["sm_mhz"] or float(peaks.get("sm_max_mhz", 2070.0))
    alu_peak = props.multi_processor_count * 128 * sm_mhz * 1e6 / 1e12
    P = wl.n_members // 2
    replay = args.hash_mode == "replay"  # the membership hash runs inside every kernel
    # algorithmic work of one update launch: a member's normal is one word of its own
    # Philox call, so each (member, noise vector) costs a whole call (80 lane-ops) plus the
    # uniform (3), transform (4) and update fma (1): 88 lane-ops per normal, P normals per
    # member (a tile shares each call among 4 elements: 28).  Replay adds the membership
    # hash of every element (one Philox call = 80 ops per 4 elements).
    ops_per_normal = 88.0
    upd_ops = ops_per_normal * P * mean_dk + (20.0 * d if replay else 0.0)
    upd_tops = upd_ops / (per["update"] * 1e-3) / 1e12
    # perturb: 6 B per member (read fp32, write bf16), 8 B for a pair perturb (two bf16
    # writes), plus 8 B of index per member for lists
    lists = args.hash_mode in ("lists", "gathered")
    pb = ((8.0 if partner is not None else 6.0) + (8.0 if lists else 0.0)) * mean_dk
    # the structural floor of a scattered pass: DRAM bytes per member it cannot avoid
    n_w = (2 if partner is not None else 1)  # working-dtype arrays the perturb writes
    floor_p = hash_sector_floor(wl.K, args.hash_mode, n_w)
    floor_r = hash_sector_floor(wl.K, args.hash_mode, 2 if args.weights == "dual" else 1)
    share = philox_block_share(torch, subs, wl.K, lists)
    value = job_throughput(world, d, args.steps, ms * 1e-3)
    out = {
        "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": (f"4B decoder-shaped bf16 set, fp32 master" if wl.name == "4b-hash" else
                                f"{wl.name}: {d} parameters in {len(wl.tensors)} tensors (profiling case)")
                               + f", K=16 hash subspaces ({args.hash_mode}), N=64 antithetic, one sweep per step",
                   "params": d, "K": wl.K, "N": wl.n_members, "sigma": wl.sigma, "alpha": wl.alpha,
                   "shaping": wl.shaping, "hash_mode": args.hash_mode, "partition_seed": wl.partition_seed,
                   "working_weights": WEIGHTS_MODES[args.weights], "l2": "inputs larger than L2, no flush"},
        "roofline": {"bound": "alu", "kernel": "update", "achieved": upd_tops, "peak": alu_peak,
                     "unit": "Tops/s", "frac": upd_tops / alu_peak, "traffic": None,
                     "peak_source": "SMs x 128 lanes x sampled SM clock",
                     "algorithmic_ops_per_launch": upd_ops},
        "kernels": {
            ("perturb_pair" if partner is not None else "perturb"): {
                "ms": per["perturb"], "launches": counts["perturb"], "GB/s": pb / (per["perturb"] * 1e-3) / 1e9,
                "frac_hbm": pb / (per["perturb"] * 1e-3) / 1e9 / hbm,
                **sector_floor_entry(floor_p, mean_dk, per["perturb"], hbm)},
            **({"perturb_partner": {"ms": per["partner"], "launches": counts["partner"]}}
               if "partner" in per else {}),
            "restore": {"ms": per["restore"], "launches": counts["restore"],
                        **sector_floor_entry(floor_r, mean_dk, per["restore"], hbm)},
            "update_fused_commit": {"ms": per["update"], "launches": counts["update"], "Tops": upd_tops,
                                    "frac_alu": upd_tops / alu_peak, "ops_per_normal": ops_per_normal,
                                    "normals_per_member": P},
            "shape": {"ms": per["shape"], "launches": counts["shape"]},
        },
        "clocks": clk,
        "e2e": None,
        "gpu_launches": sum(counts.values()),
    }
    if "mask" in per:
        out["kernels"]["mask"] = {"ms": per["mask"], "launches": counts["mask"]}
    out["philox_block_share"] = share
    print(json.dumps(out), flush=True)


def hash_sector_floor(K: int, mode: str, n_w: int) -> dict:
    """DRAM bytes per member that one pass over a hash subspace cannot avoid.  Members are
    1 element in K, each element independently, and DRAM moves 64-byte sector pairs: a
    pass that touches the members of an array of s-byte elements moves the pairs holding
    at least one member, 64 (1 - (1 - 1/K)^(64/s)) bytes per 64/s elements, i.e.
    64 (1 - (1 - 1/K)^(64/s)) / (64 / (s K)) bytes per member.  Index lists add their
    8 contiguous bytes per member; a gathered master reads theta contiguously (4 bytes);
    the replay mask adds its bits (K / 8 bytes per member).  n_w: working-dtype (bf16)
    arrays written at the members (w, and w2 or the partner buffer)."""
    q = 1.0 / K

    def scattered(s):
        m = 64 // s
        return 64.0 * (1.0 - (1.0 - q) ** m) / (m * q)

    parts = {"theta": 4.0 if mode == "gathered" else scattered(4), "w": n_w * scattered(2)}
    if mode in ("lists", "gathered"):
        parts["index"] = 8.0
    if mode == "replay-mask":
        parts["mask"] = K / 8.0
    return {"bytes_per_member": sum(parts.values()), "parts": parts}


def sector_floor_entry(floor: dict, members: float, ms: float, hbm: float) -> dict:
    gbs = floor["bytes_per_member"] * members / (ms * 1e-3) / 1e9
    return {"floor_bytes_per_member": floor["bytes_per_member"], "floor_GB/s": gbs, "frac_floor_hbm": gbs / hbm}


def philox_block_share(torch, subs, K: int, lists: bool) -> dict:
    """How often a hash subspace's consecutive members share a Philox block (the same
    g >> 2), i.e. how many Philox calls per member a gather kernel could save by reusing
    a block's words: measured on the index lists, or, for replayed subspaces, the
    expectation for independent membership, (1/4) sum_{t=0..3} (1 - (1 - 1/K)^t)."""
    if not lists:
        v = sum(1.0 - (1.0 - 1.0 / K) ** t for t in range(4)) / 4.0
        return {"value": v, "how": "expected for independent membership at this K"}
    same, pairs = 0, 0
    for sub in subs:
        q = sub.tensor >> 2
        same += int((q[1:] == q[:-1]).sum().item())
        pairs += max(q.numel() - 1, 0)
    return {"value": same / max(pairs, 1), "how": "measured on the index lists"}


def chunk_map_launches(copes, n_chunks: int) -> int:
    """Kernels one copes_random_chunk_map call launches: the keys, a bitonic sort of the
    workspace's N keys (tiles of 4,096 sorted in shared memory, then for every stage k
    above the tile one global pass per stride >= 4,096 and one tile pass), and the map."""
    import ctypes
    n = copes.load().copes_random_chunk_map_workspace_bytes(ctypes.c_uint64(n_chunks)) // 8
    tile, launches, k = 4096, 2, 8192
    while k <= n:
        launches += (k.bit_length() - 1) - (tile.bit_length() - 1) + 1
        k <<= 1
    return launches + 1


def host_link_gbs(torch, nbytes=1 << 30, reps=5):
    """Measured copy bandwidth of the host link: pinned host -> device and device -> pinned
    host, cudaMemcpyAsync of 1 GiB, best of `reps`."""
    h = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dv = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    out = {}
    for name, (dst, src) in {"h2d": (dv, h), "d2h": (h, dv)}.items():
        best = 0.0
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            dst.copy_(src, non_blocking=True)
            b.record()
            torch.cuda.synchronize()
            best = max(best, nbytes / (a.elapsed_time(b) * 1e-3) / 1e9)
        out[name] = best
    return out


def run_backup(args, wl, copes, es, torch, rank, world, local):
    """The 4B step in the CPU weight backup mode: per visit, save the subspace's context to
    pinned host memory, 32 perturbs from it, restore, shaping and the update (which
    writes the new context to both copies)."""
    from paper_2608_02391_gb300 import workloads
    layout = copes.Layout(wl.numel)
    d = wl.d
    full = make_arena(copes, torch, wl, layout)
    w = full.w
    del full
    backup = torch.empty(w.numel(), dtype=torch.bfloat16).pin_memory()
    arena = copes.BackupArena(w, backup)
    subs = es.build_subspaces(layout, "groups", wl.K, group_of=wl.group_of, tile_size=args.tile)
    for sub in subs:
        copes.backup_save(arena, sub)
    cfg = es.ESConfig(n_members=wl.n_members, sigma=wl.sigma, alpha=wl.alpha, shaping=wl.shaping)
    total = args.warmup + args.steps
    rewards = torch.from_numpy(workloads.reward_stream(wl, total * wl.K)).cuda()
    fitness = torch.empty(wl.n_members, dtype=torch.float32, device="cuda")
    # the backup mode keeps one working copy: antithetic pairs read the backup once into a
    # device partner buffer as wide as the widest subspace (unless --weights single)
    partners = [None] * wl.K if args.weights == "single" else es.Partner.per_subspace(arena, subs)

    def step(s, events=None):
        for k in range(wl.K):
            es.backup_visit(arena, subs[k], k, s, cfg, d, rewards[s * wl.K + k], fitness_out=fitness,
                            events=events, partner=partners[k])

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    copes.check()
    events = {}
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        start.record()
        for s in range(args.warmup, args.warmup + args.steps):
            step(s, events)
        end.record()
        torch.cuda.synchronize()
    ms = max_over_ranks(start.elapsed_time(end), "cuda")
    copes.check()
    if rank != 0:
        return
    link = host_link_gbs(torch)
    per = {name: float(np.mean([a.elapsed_time(b) for a, b in lst])) for name, lst in events.items()}
    counts = {name: len(lst) for name, lst in events.items()}
    mean_dk = float(np.mean([s.numel for s in subs]))
    # bytes crossing the host link per launch (bf16 = 2 B per element)
    host_bytes = {"save": 2.0, "perturb": 2.0, "restore": 2.0, "update": 4.0}
    kern = {}
    for name, hb in host_bytes.items():
        gbs = hb * mean_dk / (per[name] * 1e-3) / 1e9
        ref = link["d2h"] if name == "save" else link["h2d"]
        label = "perturb_pair" if name == "perturb" and partners[0] is not None else name
        kern[label] = {"ms": per[name], "launches": counts[name], "host_link_GB/s": gbs, "frac_link": gbs / ref}
    if "partner" in per:  # device to device, no host-link traffic
        kern["perturb_partner"] = {"ms": per["partner"], "launches": counts["partner"],
                                   "GB/s": 4.0 * mean_dk / (per["partner"] * 1e-3) / 1e9}
    kern["shape"] = {"ms": per["shape"], "launches": counts["shape"]}
    value = job_throughput(world, d, args.steps, ms * 1e-3)
    p_name = "perturb_pair" if partners[0] is not None else "perturb"
    p_gbs = kern[p_name]["host_link_GB/s"]
    out = {
        "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": ("4B decoder-shaped bf16 set, K=8 layer blocks" if wl.name == "4b" else
                                f"{wl.name}: {d} parameters in {len(wl.tensors)} tensors (profiling case), K={wl.K}")
                               + ", N=32 antithetic, CPU weight backup mode (bf16 context in pinned host memory, "
                                 "no fp32 master)",
                   "params": d, "K": wl.K, "N": wl.n_members, "tile": args.tile,
                   "working_weights": ("one bf16 copy: member 2j+1 copied in from the pair perturb's device "
                                       "partner buffer" if partners[0] is not None else WEIGHTS_MODES["single"]),
                   "l2": "inputs larger than L2, no flush"},
        "roofline": {"bound": "host_link", "kernel": p_name, "achieved": p_gbs, "peak": link["h2d"],
                     "unit": "GB/s", "frac": p_gbs / link["h2d"], "traffic": None,
                     "peak_source": "measured pinned host->device cudaMemcpyAsync of 1 GiB"},
        "host_link_measured_GB/s": link,
        "kernels": kern,
        "clocks": clocks.summary(),
        "e2e": None,
        "gpu_launches": sum(counts.values()),
    }
    print(json.dumps(out), flush=True)


def run_sync(args, wl, copes, es, torch, rank, world, local):
    """Algorithm 1 on the 4B set: per step, a fresh random-chunk partition (K = 4), the
    N_k = 8 members of every subspace perturbed under the same context, joint shaping and
    the K composed updates + commit."""
    from paper_2608_02391_gb300 import workloads
    K, chunk = 4, 65536
    layout = copes.Layout(wl.numel)
    d = wl.d
    arena = make_arena(copes, torch, wl, layout, copies=n_copies(args))
    cfg = es.ESConfig(n_members=wl.n_members, sigma=wl.sigma, alpha=wl.alpha, shaping="zscore",
                      convention=copes.COEF_PAPER, dimension_aware=True)
    total = args.warmup + args.steps
    rewards = torch.from_numpy(workloads.reward_stream(wl, total)).cuda()

    # each step's partition is built on a side stream while the previous step runs
    parts = es.ChunkPrefetcher(layout, K, lambda s: 1000 + s, chunk=chunk, tile_size=args.tile)
    # random chunks spread every subspace over the arena: one partner buffer covers it
    if args.weights == "quad":
        partner = es.Partner.four_copies(arena)
    elif args.weights == "dual":
        partner = es.Partner.second_copy(arena)
    elif args.weights == "partner":
        partner = es.Partner(torch.empty(layout.d_pad, dtype=arena.w.dtype, device="cuda"), 0)
    else:
        partner = None

    def step(s, events=None):
        subs = parts.take(s, events=events)
        es.sync_step(arena, subs, s, cfg, d, rewards[s], joint=True, events=events, partner=partner)
        if s + 1 < total:
            parts.prefetch(s + 1, events=events)
        return subs

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    copes.check()
    events = {}
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        start.record()
        for s in range(args.warmup, args.warmup + args.steps):
            subs = step(s, events)
        end.record()
        torch.cuda.synchronize()
    ms = max_over_ranks(start.elapsed_time(end), "cuda")
    copes.check()
    if rank != 0:
        return
    per = {name: float(np.mean([a.elapsed_time(b) for a, b in lst])) for name, lst in events.items()}
    counts = {name: len(lst) for name, lst in events.items()}
    mean_dk = float(np.mean([s.numel for s in subs]))
    peaks, _ = measured_peaks()
    hbm = float(peaks["hbm_gbs"])
    clk = clocks.summary()
    sm_mhz = clk["sm_mhz"] or 2070.0
    props = torch.cuda.get_device_properties(local)
    alu_peak = props.multi_processor_count * 128 * sm_mhz * 1e6 / 1e12
    P = (wl.n_members // K) // 2
    upd_tops = 28.0 * P * mean_dk / (per["update"] * 1e-3) / 1e12
    upd_bytes = 8.0 + 2.0 * n_copies(args)  # read and write theta, write every working copy
    upd_gbs = upd_bytes * mean_dk / (per["update"] * 1e-3) / 1e9
    # the update's roofline is the slower of its ALU and HBM bounds
    t_alu = 28.0 * P * mean_dk / (alu_peak * 1e12)
    t_hbm = upd_bytes * mean_dk / (hbm * 1e9)
    pk = perturb_kernel(args)
    perturb_gbs = {"perturb_two_pairs": 12.0, "perturb_pair": 8.0, "perturb": 6.0}[pk] * mean_dk / (per["perturb"] * 1e-3) / 1e9
    value = job_throughput(world, d, args.steps, ms * 1e-3)
    out = {
        "metric": METRIC, "value": value, "unit": "params/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "4B decoder-shaped bf16 set, fp32 master, Algorithm 1: K=4 random chunks "
                               "(65,536) resampled per step, N=32 antithetic (N_k=8), dimension-aware sigma_k, "
                               "joint z-score, coefficient alpha/N_k",
                   "params": d, "K": K, "N": wl.n_members, "chunk": chunk, "sigma": wl.sigma, "alpha": wl.alpha,
                   "tile": args.tile, "working_weights": WEIGHTS_MODES[args.weights],
                   "l2": "inputs larger than L2, no flush"},
        "roofline": {"bound": "hbm", "kernel": pk, "achieved": perturb_gbs,
                     "peak": hbm, "unit": "GB/s", "frac": perturb_gbs / hbm, "traffic": None,
                     "peak_source": "measured"},
        "kernels": {
            "partition": {"ms": per.get("partition"), "launches": counts.get("partition", 0),
                          "note": "side-stream window, host tile building included; overlapped with "
                                  "the previous step"},
            pk: {"ms": per["perturb"], "launches": counts["perturb"], "GB/s": perturb_gbs,
                 "frac_hbm": perturb_gbs / hbm},
            **({"perturb_partner": {"ms": per["partner"], "launches": counts["partner"],
                                    "GB/s": 4.0 * mean_dk / (per["partner"] * 1e-3) / 1e9}}
               if "partner" in per else {}),
            "restore": {"ms": per["restore"], "launches": counts["restore"],
                        "GB/s": (4.0 + 2.0 * n_copies(args)) * mean_dk / (per["restore"] * 1e-3) / 1e9},
            "update_fused_commit": {"ms": per["update"], "launches": counts["update"], "Tops": upd_tops,
                                    "GB/s": upd_gbs, "normals_per_elem": P,
                                    "frac_of_slower_bound": max(t_alu, t_hbm) / (per["update"] * 1e-3),
                                    "bound": "alu" if t_alu >= t_hbm else "hbm"},
            "shape": {"ms": per["shape"], "launches": counts["shape"]},
        },
        "clocks": clk,
        "e2e": None,
        # each timed partition build launches the random-chunk map's kernels (keys, bitonic
        # sort, map); its tile tables (over 1,000 ranges each) are copied, not launched
        "gpu_launches": sum(v for k, v in counts.items() if k != "partition")
        + counts.get("partition", 0) * chunk_map_launches(copes, -(-layout.d_pad // chunk)),
    }
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
