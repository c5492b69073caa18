"""Host-side schedules of the CoPES ES core (orchestration only; every step is a library
kernel launched through the ``copes`` binding).

round_robin_visit  one ES iteration on one subspace: N perturbed evaluations, restore,
                   shaping, fused update + context commit (the cooperative-coevolution
                   visit; one "cycle" visits k = 0 .. K-1 in order).
sync_step          one CoPES training step (Algorithm 1): every subspace's N_k = N / K
                   members are evaluated under the same pre-update context, rewards are
                   standardised jointly (Eq. 12) or per subspace (Sec. 4.4 ablation), and
                   all K subspace updates are composed (Eq. 13) before the commit.
backup_visit       round_robin_visit in the CPU weight backup mode (Supp. A.8): the
                   context is saved to pinned host memory, members are perturbed from
                   it, and restore copies it back; no fp32 master.
ChunkPrefetcher    the random-chunk partition of the next sync_step built on a side stream
                   while the current step's kernels run (Algorithm 1 resamples it every
                   step).
state_dict /       the resumable state (fp32 master, ES configuration, next iteration):
load_state         noise is counter-based, so resuming from it is bit-exact.
population_visit   round_robin_visit with the population split across the ranks of a
                   process group, each rank holding a full replica of theta: a rank
                   evaluates its slice of the members, the N reward scalars are
                   all-gathered on the host, and every rank applies the same update, so
                   the replicas stay bit-identical (the paper's population-parallel ES
                   layout, Sec. 3.3 seed replay: only seeds and scalar rewards travel).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Callable, List, Optional, Sequence

import numpy as np
import torch

from . import copes


@dataclass
class ESConfig:
    n_members: int
    sigma: float
    alpha: float
    shaping: str = "zscore"
    pairing: int = copes.ANTITHETIC
    convention: int = copes.COEF_OPENAI
    dimension_aware: bool = False
    base_seed: int = 33


@dataclass
class Partner:
    """Buffer for the antithetic partner's weights (copes_perturb_pair): element g of the
    arena at buf[g - base], in the working dtype.  Partner.covering(arena, subs) sizes one
    for every element of `subs`.  in_place: the buffer is the arena's second working
    buffer w2 (Partner.second_copy), so the partner member is evaluated there directly and
    nothing is copied.  two_pairs: the arena has four working copies
    (Partner.four_copies), and two consecutive antithetic pairs with the same sign order
    are written to w, w2, w3 and w4 by one copes_perturb_two_pairs."""
    buf: torch.Tensor
    base: int
    in_place: bool = False
    two_pairs: bool = False

    @classmethod
    def second_copy(cls, arena: copes.Arena) -> "Partner":
        """The arena's second working buffer as the partner: member 2j is evaluated on w,
        member 2j + 1 on w2."""
        assert arena.w2 is not None, "the arena has no second working buffer"
        return cls(arena.w2, 0, True)

    @classmethod
    def four_copies(cls, arena: copes.Arena) -> "Partner":
        """Members 4m .. 4m + 3 (noise vectors 2m and 2m + 1, signs +, -, +, -) evaluated
        on w, w2, w3 and w4, all four written by one pass; a pair left over at the end of
        the member list goes to w and w2."""
        assert arena.w4 is not None, "the arena has no four working copies"
        return cls(arena.w2, 0, True, True)

    @classmethod
    def covering(cls, arena: copes.Arena, subs: Sequence[copes.SubspaceHandle]) -> "Partner":
        """One buffer covering every element of `subs` (for steps that perturb them all,
        e.g. sync_step)."""
        buf, base = copes.partner_buffer(arena, subs)
        return cls(buf, base)

    @classmethod
    def per_subspace(cls, arena: copes.Arena, subs: Sequence[copes.SubspaceHandle]) -> List["Partner"]:
        """One buffer as wide as the widest subspace's span, shared by a Partner per
        subspace with that subspace's own base (round-robin visits use one at a time)."""
        spans = copes.subspace_spans(arena, subs)
        width = max((hi - lo for lo, hi in spans), default=0)
        buf = torch.empty(max(width, 8), dtype=arena.w.dtype, device=arena.w.device)
        return [cls(buf, lo) for lo, _ in spans]


def _antithetic(nid, sign, a: int, b: int) -> bool:
    """Members a and b share a noise vector with opposite signs."""
    return nid[b] == nid[a] and sign[b] == -sign[a]


def perturb_members(arena: copes.Arena, sub: copes.SubspaceHandle, members: Sequence[int], nid, sign,
                    seeds, s_k: float, live: Callable[[int], None], partner: Optional[Partner] = None,
                    events: Optional[dict] = None, backup: bool = False) -> None:
    """Perturbs each member of `members` in order (Eq. 8) and calls live(i) while member i's
    perturbation is in place (in arena.live).  With a partner buffer, a member whose
    successor shares its noise vector with the opposite sign (an antithetic pair) is
    perturbed by copes_perturb_pair, and the successor's weights are then copied in from
    the buffer, or, for an in-place partner (the arena's w2), evaluated there: one noise
    generation per pair, bit-identical weights.  With four working copies
    (Partner.four_copies), two such pairs in a row whose first members have the same sign
    are written to w, w2, w3 and w4 by one copes_perturb_two_pairs and evaluated there
    (TILES subspaces; other kinds take the pairs one at a time).
    backup: the CPU weight backup mode's calls (arena is a copes.BackupArena)."""
    if backup:
        assert partner is None or not partner.two_pairs, "the backup mode has one working copy"
        perturb, pair, copy = copes.backup_perturb, copes.backup_perturb_pair, copes.backup_perturb_partner
    else:
        perturb, pair, copy = copes.perturb, copes.perturb_pair, copes.perturb_partner
    staged = None  # the member whose weights the partner buffer holds
    ready = {}     # member -> the working copy that already holds its weights
    for pos, i in enumerate(members):
        nxt = members[pos + 1] if pos + 1 < len(members) else None
        seed, ss = int(seeds[nid[i]]), float(sign[i]) * s_k
        where = None if arena is None else arena.w
        quad = (members[pos:pos + 4] if partner is not None and partner.two_pairs
                and sub.kind == copes.SUBSPACE_TILES else [])
        if i in ready:
            where = ready.pop(i)
        elif staged == i and partner.in_place:
            where = partner.buf
        elif staged == i:
            _timed(events, "partner", lambda: copy(arena, sub, partner.buf, partner.base))
        elif (len(quad) == 4 and _antithetic(nid, sign, quad[0], quad[1]) and _antithetic(nid, sign, quad[2], quad[3])
              and sign[quad[2]] == sign[i]):
            seed_b = int(seeds[nid[quad[2]]])
            _timed(events, "perturb", lambda: copes.perturb_two_pairs(arena, sub, seed, seed_b, ss))
            ready = {quad[1]: arena.w2, quad[2]: arena.w3, quad[3]: arena.w4}
        elif partner is not None and nxt is not None and _antithetic(nid, sign, i, nxt):
            _timed(events, "perturb", lambda: pair(arena, sub, seed, ss, partner.buf, partner.base))
            staged = nxt
        else:
            _timed(events, "perturb", lambda: perturb(arena, sub, seed, ss))
        if arena is not None:
            arena.live = where
        live(i)
    if arena is not None:
        arena.live = arena.w


def sigma_k(cfg: ESConfig, d: int, d_k: int) -> float:
    """Eq. 11 when dimension-aware, else the configured sigma."""
    return copes.sigma_eff(cfg.sigma, d, d_k, cfg.dimension_aware)


def round_robin_visit(arena: copes.Arena, sub: copes.SubspaceHandle, k: int, iteration: int,
                      cfg: ESConfig, d: int, rewards: torch.Tensor,
                      evaluate: Optional[Callable[[int], None]] = None,
                      fitness_out: Optional[torch.Tensor] = None,
                      events: Optional[dict] = None, partner: Optional[Partner] = None) -> torch.Tensor:
    """One ES iteration on subspace k.  `rewards` (device fp32 [N]) holds the members'
    rewards; `evaluate(i)` runs while member i's perturbation is live (it may write
    rewards[i]).  `partner`: perturb antithetic pairs with one noise generation
    (perturb_members).  Returns the shaped fitness."""
    nid, sign, P = copes.member_table(cfg.n_members, cfg.pairing)
    seeds = copes.member_seeds(cfg.base_seed, iteration, k, P)
    s_k = sigma_k(cfg, d, sub.numel)
    perturb_members(arena, sub, range(cfg.n_members), nid, sign, seeds, s_k,
                    evaluate if evaluate is not None else (lambda i: None), partner, events)
    _timed(events, "restore", lambda: copes.restore(arena, sub))
    f = fitness_out if fitness_out is not None else torch.empty_like(rewards)
    _timed(events, "shape", lambda: copes.shape_fitness(rewards, cfg.shaping, out=f))
    coef = copes.step_coef(cfg.alpha, cfg.n_members, s_k, cfg.convention)
    _timed(events, "update", lambda: copes.update(arena, sub, nid, sign, f, seeds, coef, fuse_commit=True))
    return f


def backup_visit(arena: copes.BackupArena, sub: copes.SubspaceHandle, k: int, iteration: int,
                 cfg: ESConfig, d: int, rewards: torch.Tensor,
                 evaluate: Optional[Callable[[int], None]] = None,
                 fitness_out: Optional[torch.Tensor] = None,
                 events: Optional[dict] = None, partner: Optional[Partner] = None) -> torch.Tensor:
    """One ES iteration on subspace k in the CPU weight backup mode: save the context of S
    to the host backup, evaluate the N members perturbed from it, restore, shape, and
    apply the update, which writes the new context to the weights and the backup.
    `partner` (a device buffer, not in place): antithetic pairs read the backup once."""
    assert partner is None or not partner.in_place, "the backup mode has one working copy"
    nid, sign, P = copes.member_table(cfg.n_members, cfg.pairing)
    seeds = copes.member_seeds(cfg.base_seed, iteration, k, P)
    s_k = sigma_k(cfg, d, sub.numel)
    _timed(events, "save", lambda: copes.backup_save(arena, sub))
    perturb_members(arena, sub, range(cfg.n_members), nid, sign, seeds, s_k,
                    evaluate if evaluate is not None else (lambda i: None), partner, events, backup=True)
    _timed(events, "restore", lambda: copes.backup_restore(arena, sub))
    f = fitness_out if fitness_out is not None else torch.empty_like(rewards)
    _timed(events, "shape", lambda: copes.shape_fitness(rewards, cfg.shaping, out=f))
    coef = copes.step_coef(cfg.alpha, cfg.n_members, s_k, cfg.convention)
    _timed(events, "update", lambda: copes.backup_update(arena, sub, nid, sign, f, seeds, coef))
    return f


def sync_step(arena: copes.Arena, subs: Sequence[copes.SubspaceHandle], iteration: int,
              cfg: ESConfig, d: int, rewards: torch.Tensor,
              evaluate: Optional[Callable[[int, int], None]] = None,
              joint: bool = True, events: Optional[dict] = None,
              partner: Optional[Partner] = None) -> torch.Tensor:
    """Algorithm 1: N = cfg.n_members split into N_k = N / K per subspace; rewards is the
    device fp32 [N] vector laid out subspace by subspace (member i of subspace k at
    k N_k + i).  evaluate(k, i) runs while that member's perturbation is live.  `partner`
    (covering every subspace): antithetic pairs with one noise generation."""
    K = len(subs)
    if cfg.n_members % K:
        raise ValueError("N must be divisible by K (Sec. 3.2)")
    n_k = cfg.n_members // K
    nid, sign, P = copes.member_table(n_k, cfg.pairing)
    seeds = [copes.member_seeds(cfg.base_seed, iteration, k, P) for k in range(K)]
    for k, sub in enumerate(subs):
        s_k = sigma_k(cfg, d, sub.numel)
        perturb_members(arena, sub, range(n_k), nid, sign, seeds[k], s_k,
                        (lambda i: evaluate(k, i)) if evaluate is not None else (lambda i: None),
                        partner, events)
        # the next subspace is evaluated under the same context
        _timed(events, "restore", lambda: copes.restore(arena, sub))
    if joint:
        f = _timed(events, "shape", lambda: copes.shape_fitness(
            rewards, copes.SHAPE_ZSCORE if cfg.shaping == "zscore" else cfg.shaping))
    else:
        group = torch.arange(cfg.n_members, device=rewards.device, dtype=torch.int32) // n_k
        f = _timed(events, "shape", lambda: copes.shape_fitness(rewards, copes.SHAPE_ZSCORE_GROUPED, group=group))
    for k, sub in enumerate(subs):  # every g_k from the same pre-update theta (disjoint supports)
        s_k = sigma_k(cfg, d, sub.numel)
        coef = copes.step_coef(cfg.alpha, n_k, s_k, cfg.convention)
        _timed(events, "update", lambda: copes.update(arena, sub, nid, sign, f[k * n_k:(k + 1) * n_k], seeds[k],
                                                      coef, fuse_commit=True))
    return f


def _timed(events: Optional[dict], name: str, fn):
    if events is None:
        return fn()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record()
    out = fn()
    end.record()
    events.setdefault(name, []).append((start, end))
    return out


def build_subspaces(layout: copes.Layout, mode: str, K: int, group_of: Optional[List[int]] = None,
                    seed: int = 0, chunk: int = 65536, tile_size: int = copes.DEFAULT_TILE):
    """All K subspaces of a partition (tiles for range modes, index lists for hash)."""
    if mode == "hash":
        return copes.hash_partition(layout, K, seed)
    if mode == "contiguous":
        return [copes.subspace_build(layout, copes.PART_CONTIGUOUS, K, k, tile_size=tile_size) for k in range(K)]
    if mode == "groups":
        return [copes.subspace_build(layout, copes.PART_TENSOR_GROUPS, K, k, group_of=group_of,
                                     tile_size=tile_size) for k in range(K)]
    if mode == "random_chunks":
        n_chunks = (layout.d_pad + chunk - 1) // chunk
        cmap = copes.random_chunk_map(n_chunks, K, seed)
        return [copes.subspace_build(layout, copes.PART_RANDOM_CHUNKS, K, k, seed=seed, chunk=chunk,
                                     chunk_map=cmap, tile_size=tile_size) for k in range(K)]
    raise ValueError(mode)


class ChunkPrefetcher:
    """Random equal-size chunk partitions (Algorithm 1 resamples the partition every step,
    Sec. 3.2), each built one step ahead on a side stream.

    Building a partition copies the device chunk map to the host and synchronises the
    stream it runs on before the host writes the tile tables.  On a side stream that
    wait covers only the map's own kernels, so the host builds step s + 1's tables while
    the main stream still executes step s, and the copy engines move them meanwhile.
    take(s) makes the caller's stream wait for step s's build and records the tables'
    use on that stream, so the caching allocator keeps them until its kernels are done.
    """

    def __init__(self, layout: copes.Layout, K: int, seed_of: Callable[[int], int], chunk: int = 65536,
                 tile_size: int = copes.DEFAULT_TILE, device="cuda"):
        self.layout, self.K, self.seed_of = layout, K, seed_of
        self.chunk, self.tile_size = chunk, tile_size
        self.side = torch.cuda.Stream(device=device)
        self.ready = {}

    def _build(self, step: int, events: Optional[dict] = None):
        start = end = None
        if events is not None:
            start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        done = torch.cuda.Event()
        with torch.cuda.stream(self.side):
            if start is not None:
                start.record(self.side)
            subs = build_subspaces(self.layout, "random_chunks", self.K, seed=self.seed_of(step),
                                   chunk=self.chunk, tile_size=self.tile_size)
            if end is not None:
                end.record(self.side)
                events.setdefault("partition", []).append((start, end))
            done.record(self.side)
        return subs, done

    def prefetch(self, step: int, events: Optional[dict] = None) -> None:
        if step not in self.ready:
            self.ready[step] = self._build(step, events)

    def take(self, step: int, stream: Optional[torch.cuda.Stream] = None,
             events: Optional[dict] = None) -> List[copes.SubspaceHandle]:
        subs, done = self.ready.pop(step, None) or self._build(step, events)
        stream = stream or torch.cuda.current_stream()
        stream.wait_event(done)
        for sub in subs:
            sub.tensor.record_stream(stream)
        return subs


# ------------------------------------------------------------- population parallelism
def member_slice(rank: int, world: int, n_members: int) -> range:
    """The members rank `rank` evaluates: consecutive blocks of ceil(N / world)."""
    m = -(-n_members // world)
    return range(min(rank * m, n_members), min((rank + 1) * m, n_members))


def gather_rewards(local: np.ndarray, n_members: int, group=None) -> np.ndarray:
    """All-gather of the members' rewards over `group` (host tensors; gloo or any backend
    that gathers CPU tensors).  `local` is a float32 [N] array in which this rank has
    written the rewards of member_slice(rank, world, N); the result is the full [N] vector,
    identical on every rank and equal bit for bit to each slice's source values."""
    import torch.distributed as dist
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    m = -(-n_members // world)
    mine = member_slice(rank, world, n_members)
    buf = torch.zeros(m, dtype=torch.float32)
    buf[:len(mine)] = torch.from_numpy(np.ascontiguousarray(local[mine.start:mine.stop], np.float32))
    parts = [torch.empty(m, dtype=torch.float32) for _ in range(world)]
    dist.all_gather(parts, buf, group=group)
    return torch.cat(parts)[:n_members].numpy()


def population_visit(arena: copes.Arena, sub: copes.SubspaceHandle, k: int, iteration: int,
                     cfg: ESConfig, d: int, evaluate: Callable[[int], float], group=None,
                     fitness_out: Optional[torch.Tensor] = None,
                     partner: Optional[Partner] = None,
                     rewards_out: Optional[np.ndarray] = None) -> torch.Tensor:
    """One ES iteration on subspace k, population-parallel over the ranks of `group`.
    Every rank holds the same theta; rank r evaluates members member_slice(r, R, N):
    perturb, evaluate(i) -> reward (host float) while the perturbation is live, and
    restores S afterwards.  The rewards are all-gathered, then every rank shapes the same
    vector and applies the same fused update + commit, so the replicas stay identical.
    rewards_out (host float32 [N]) receives the gathered rewards."""
    import torch.distributed as dist
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    N = cfg.n_members
    nid, sign, P = copes.member_table(N, cfg.pairing)
    seeds = copes.member_seeds(cfg.base_seed, iteration, k, P)
    s_k = sigma_k(cfg, d, sub.numel)
    local = np.zeros(N, np.float32)

    def live(i):
        local[i] = np.float32(evaluate(i))

    perturb_members(arena, sub, member_slice(rank, world, N), nid, sign, seeds, s_k, live, partner)
    copes.restore(arena, sub)
    gathered = gather_rewards(local, N, group)
    if rewards_out is not None:
        rewards_out[:] = gathered
    rewards = torch.from_numpy(gathered).to(arena.w.device)
    f = fitness_out if fitness_out is not None else torch.empty_like(rewards)
    copes.shape_fitness(rewards, cfg.shaping, out=f)
    coef = copes.step_coef(cfg.alpha, N, s_k, cfg.convention)
    copes.update(arena, sub, nid, sign, f, seeds, coef, fuse_commit=True)
    return f


# ------------------------------------------------------------------ checkpoint / resume
def state_dict(arena: copes.Arena, cfg: ESConfig, next_iteration: int, **extra) -> dict:
    """The resumable ES state: the fp32 master (host copy), the configuration, the next
    iteration index and how many working copies the arena keeps (1, 2 or 4).  Member seeds
    and noise are functions of (base seed, iteration, subspace, member) and (seed, index),
    and partition seeds are part of `extra`, so nothing else needs saving: a run resumed
    from this state continues bit for bit.  The working copies are not saved: between ES
    iterations all of them equal round(theta) and are rebuilt from the master."""
    return {"master": arena.master.detach().cpu().clone(), "working_dtype": str(arena.w.dtype),
            "working_copies": len(arena.copies), "config": dict(cfg.__dict__),
            "next_iteration": int(next_iteration), **extra}


def load_state(state: dict, device="cuda") -> tuple:
    """Rebuilds (arena, cfg, next_iteration) from state_dict's output: the master is
    copied to the device and the saved number of working copies is committed from it
    (every copy = round(theta) over the whole arena)."""
    master = state["master"].to(device).contiguous()
    dtype = {"torch.bfloat16": torch.bfloat16, "torch.float32": torch.float32}[state["working_dtype"]]
    n = master.numel()
    n_copies = int(state.get("working_copies", 1))
    assert n_copies in (1, 2, 4), f"{n_copies} working copies"
    copies = [torch.empty(n, dtype=dtype, device=device) for _ in range(n_copies)]
    arena = copes.Arena(copies[0], master, *copies[1:])
    everything = copes.tiles_from_ranges([(0, n)], device=device)
    copes.context_commit(arena, everything)  # commit writes every working copy
    return arena, ESConfig(**state["config"]), state["next_iteration"]
