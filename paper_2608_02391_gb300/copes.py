"""Thin ctypes binding of libcopes.so (the C ABI in include/copes.h).

Argument marshalling only: torch supplies device memory and streams, every step runs in
the library's CUDA kernels.  The names follow the C ABI.  Loading fails loudly when the
library has not been built; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import List, Optional, Sequence, Tuple

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libcopes.so")

OK = 0
ERR_INVALID_ARG, ERR_ALIGNMENT, ERR_SIZE, ERR_WORKSPACE, ERR_CUDA, ERR_DEVICE_CHECK, ERR_UNSUPPORTED = \
    -1, -2, -3, -4, -5, -6, -7
BF16, FP32 = 0, 1
TAG_NOISE, TAG_INIT, TAG_PARTITION, TAG_SEED, TAG_CHUNK = 0, 1, 2, 3, 4
MAX_MEMBERS, MAX_NOISE, MAX_K, TILE_MAX = 256, 256, 64, 1 << 20
SUBSPACE_TILES, SUBSPACE_INDICES, SUBSPACE_HASH_REPLAY = 0, 1, 2
PART_CONTIGUOUS, PART_TENSOR_GROUPS, PART_HASH, PART_RANDOM_CHUNKS = 0, 1, 2, 3
SHAPE_NONE, SHAPE_ZSCORE, SHAPE_ZSCORE_GROUPED, SHAPE_CENTERED_RANK = 0, 1, 2, 3
ONE_SIDED, ANTITHETIC = 0, 1
COEF_PAPER, COEF_OPENAI = 0, 1
DEFAULT_TILE = 1 << 14

SHAPE_MODES = {"none": SHAPE_NONE, "zscore": SHAPE_ZSCORE, "zscore_grouped": SHAPE_ZSCORE_GROUPED,
               "centered_rank": SHAPE_CENTERED_RANK}


class CopesError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"[{code}] {message}")
        self.code = code


class Params(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("master", ctypes.c_void_p), ("n_alloc", ctypes.c_uint64),
                ("dtype", ctypes.c_int), ("w2", ctypes.c_void_p), ("w3", ctypes.c_void_p),
                ("w4", ctypes.c_void_p)]


class Subspace(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("tiles", ctypes.c_void_p), ("n_tiles", ctypes.c_uint64),
                ("index", ctypes.c_void_p), ("n_index", ctypes.c_uint64),
                ("replay", ctypes.c_void_p), ("n_replay_tiles", ctypes.c_uint64),
                ("n_replay_tensors", ctypes.c_int), ("K", ctypes.c_int), ("k", ctypes.c_int),
                ("seed", ctypes.c_uint64), ("gathered", ctypes.c_void_p), ("replay_mask", ctypes.c_void_p)]


class BackupParams(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("backup", ctypes.c_void_p), ("n_alloc", ctypes.c_uint64)]


class LayoutDesc(ctypes.Structure):
    _fields_ = [("n_tensors", ctypes.c_int), ("numel", ctypes.c_void_p), ("tensor_id", ctypes.c_void_p)]


class PartitionSpec(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int), ("K", ctypes.c_int), ("seed", ctypes.c_uint64),
                ("chunk", ctypes.c_uint64), ("group_of", ctypes.c_void_p)]


_lib = None

# name -> (restype, argtypes); every function declared in include/copes.h.
_VP, _U64, _U32, _I32, _F32, _F64, _SZ = (ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint32,
                                          ctypes.c_int, ctypes.c_float, ctypes.c_double,
                                          ctypes.c_size_t)
SIGNATURES = {
    "copes_version": (ctypes.c_char_p, []),
    "copes_last_error": (_I32, [_VP, _SZ]),
    "copes_check": (_I32, [_VP]),
    "copes_layout": (_I32, [_VP, _VP]),
    "copes_sigma_eff": (_F64, [_F64, _F64, _F64, _I32]),
    "copes_step_coef": (_F64, [_F64, _I32, _F64, _I32]),
    "copes_member_table": (_I32, [_I32, _I32, _VP, _VP]),
    "copes_member_seed": (_U64, [_U64, _U32, _U32, _U32]),
    "copes_subspace_build": (_I32, [_VP, _VP, _I32, _U64, _VP, _VP, _U64, _VP, _VP]),
    "copes_tiles_from_ranges": (_I32, [_VP, _VP, _I32, _U64, _VP, _U64, _VP, _VP]),
    "copes_random_chunk_map_workspace_bytes": (_SZ, [_U64]),
    "copes_random_chunk_map": (_I32, [_U64, _I32, _U64, _VP, _VP, _SZ, _VP]),
    "copes_hash_workspace_bytes": (_SZ, [_VP, _I32]),
    "copes_hash_count": (_I32, [_VP, _I32, _U64, _VP, _SZ, _VP, _VP]),
    "copes_hash_fill": (_I32, [_VP, _I32, _U64, _VP, _SZ, _VP, _VP]),
    "copes_hash_partition_static": (_I32, [_VP, _I32, _U64, _VP, _VP, _VP, _VP]),
    "copes_hash_replay_bytes": (_SZ, [_VP]),
    "copes_hash_replay_subspace": (_I32, [_VP, _I32, _U64, _I32, _VP, _SZ, _VP, _VP]),
    "copes_perturb": (_I32, [_VP, _VP, _U64, _F32, _VP]),
    "copes_perturb_pair": (_I32, [_VP, _VP, _U64, _F32, _VP, _U64, _U64, _VP]),
    "copes_perturb_partner": (_I32, [_VP, _VP, _VP, _U64, _U64, _VP]),
    "copes_perturb_two_pairs": (_I32, [_VP, _VP, _U64, _U64, _F32, _VP]),
    "copes_restore": (_I32, [_VP, _VP, _VP]),
    "copes_context_commit": (_I32, [_VP, _VP, _VP]),
    "copes_shape_fitness": (_I32, [_VP, _I32, _VP, _I32, _VP, _VP]),
    "copes_update": (_I32, [_VP, _VP, _I32, _VP, _VP, _VP, _I32, _VP, _F32, _I32, _VP]),
    "copes_init_normal": (_I32, [_VP, _VP, _U64, _F32, _F32, _VP]),
    "copes_gather_master": (_I32, [_VP, _VP, _VP]),
    "copes_hash_replay_mask": (_I32, [_VP, _VP, _VP]),
    "copes_scatter_master": (_I32, [_VP, _VP, _VP]),
    "copes_backup_save": (_I32, [_VP, _VP, _VP]),
    "copes_backup_perturb": (_I32, [_VP, _VP, _U64, _F32, _VP]),
    "copes_backup_perturb_pair": (_I32, [_VP, _VP, _U64, _F32, _VP, _U64, _U64, _VP]),
    "copes_backup_perturb_partner": (_I32, [_VP, _VP, _VP, _U64, _U64, _VP]),
    "copes_backup_restore": (_I32, [_VP, _VP, _VP]),
    "copes_backup_update": (_I32, [_VP, _VP, _I32, _VP, _VP, _VP, _I32, _VP, _F32, _VP]),
    "copes_debug_philox": (_I32, [_U64, _U64, _U64, _U32, _U32, _VP, _VP]),
    "copes_debug_normals": (_I32, [_U64, _U32, _U64, _U64, _VP, _VP]),
    "copes_debug_transform": (_I32, [_VP, _U64, _VP, _VP]),
}


def load():
    """Load libcopes.so (raises if it is missing: build it with __graft_entry__.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build the CUDA library first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def last_error() -> str:
    buf = ctypes.create_string_buffer(1024)
    load().copes_last_error(buf, len(buf))
    return buf.value.decode()


def _check(rc: int) -> int:
    if rc < 0:
        raise CopesError(rc, last_error())
    return rc


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _np_ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


# ------------------------------------------------------------------------ host helpers
def version() -> str:
    return load().copes_version().decode()


def check(stream=None) -> None:
    """Synchronise the stream and raise if a kernel's range check fired."""
    _check(load().copes_check(_stream(stream)))


def sigma_eff(sigma: float, d: float, d_k: float, dimension_aware: bool = True) -> float:
    return load().copes_sigma_eff(sigma, float(d), float(d_k), int(dimension_aware))


def step_coef(alpha: float, n_members: int, sigma_eff_: float, convention: int) -> float:
    return load().copes_step_coef(alpha, n_members, sigma_eff_, convention)


def member_table(n_members: int, pairing: int):
    nid = np.zeros(n_members, np.int32)
    sign = np.zeros(n_members, np.int8)
    P = _check(load().copes_member_table(n_members, pairing, _np_ptr(nid), _np_ptr(sign)))
    return nid, sign, P


def member_seed(base_seed: int, iteration: int, k: int, j: int) -> int:
    return int(load().copes_member_seed(base_seed, iteration, k, j))


def member_seeds(base_seed: int, iteration: int, k: int, n_noise: int) -> np.ndarray:
    return np.array([member_seed(base_seed, iteration, k, j) for j in range(n_noise)], np.uint64)


class Layout:
    """Host view of a tensor table (copes_layout_desc); keeps its arrays alive."""

    def __init__(self, numel: Sequence[int], tensor_id: Optional[Sequence[int]] = None):
        self.numel = np.ascontiguousarray(numel, dtype=np.uint64)
        self.tensor_id = None if tensor_id is None else np.ascontiguousarray(tensor_id, np.uint32)
        self.desc = LayoutDesc(self.numel.size, _np_ptr(self.numel), _np_ptr(self.tensor_id))
        self.offsets = np.zeros(self.numel.size + 1, np.uint64)
        _check(load().copes_layout(ctypes.byref(self.desc), _np_ptr(self.offsets)))

    @property
    def d_pad(self) -> int:
        return int(self.offsets[-1])


# ----------------------------------------------------------------------------- arena
class Arena:
    """The flat parameter arena: working weights w (bf16 or fp32) and the fp32 master, and
    optionally further working copies -- w2 (copes_params.w2), or w2, w3 and w4 -- that
    restore, commit and init keep equal to w outside the live members' perturbations.
    `live` is the working buffer that holds the member being evaluated (w, or the copy a
    pair's or two pairs' perturb wrote that member to)."""

    def __init__(self, w: torch.Tensor, master: torch.Tensor, w2: Optional[torch.Tensor] = None,
                 w3: Optional[torch.Tensor] = None, w4: Optional[torch.Tensor] = None):
        assert w.is_cuda and master.is_cuda and w.is_contiguous() and master.is_contiguous()
        assert master.dtype == torch.float32 and w.numel() == master.numel()
        assert (w3 is None) == (w4 is None) and (w3 is None or w2 is not None), \
            "w3 and w4 come together, and only with w2"
        for c in (w2, w3, w4):
            if c is not None:
                assert c.is_cuda and c.is_contiguous() and c.dtype == w.dtype and c.numel() == w.numel()
        self.w, self.master, self.w2, self.w3, self.w4 = w, master, w2, w3, w4
        self.live = w
        dt = {torch.bfloat16: BF16, torch.float32: FP32}[w.dtype]
        ptr = lambda c: None if c is None else c.data_ptr()
        self.params = Params(w.data_ptr(), master.data_ptr(), w.numel(), dt, ptr(w2), ptr(w3), ptr(w4))

    @property
    def copies(self) -> List[torch.Tensor]:
        """The working copies in order: [w], [w, w2] or [w, w2, w3, w4]."""
        return [c for c in (self.w, self.w2, self.w3, self.w4) if c is not None]

    @classmethod
    def empty(cls, n: int, dtype=torch.bfloat16, device="cuda"):
        return cls(torch.empty(n, dtype=dtype, device=device), torch.empty(n, dtype=torch.float32, device=device))

    @property
    def n_alloc(self) -> int:
        return self.w.numel()


@dataclass
class SubspaceHandle:
    """A subspace: device tiles ([n, 2] int64 holding uint64 bounds), a device index list, or
    a hash-replay subspace (tensor = its device tensor table, replay = the filled struct)."""
    kind: int
    tensor: torch.Tensor
    numel: int
    replay: Optional[Subspace] = None
    gathered: Optional[torch.Tensor] = None  # INDICES: theta in list order (gather_master)
    mask: Optional[torch.Tensor] = None      # HASH_REPLAY: membership bits (hash_replay_mask)

    def struct(self) -> Subspace:
        if self.kind == SUBSPACE_HASH_REPLAY:
            return self.replay
        if self.kind == SUBSPACE_TILES:
            return Subspace(SUBSPACE_TILES, self.tensor.data_ptr() if self.tensor.numel() else None,
                            self.tensor.shape[0], None, 0)
        S = Subspace(SUBSPACE_INDICES, None, 0, self.tensor.data_ptr() if self.tensor.numel() else None,
                     self.tensor.numel())
        if self.gathered is not None:
            S.gathered = self.gathered.data_ptr()
        return S


def _tiles_result(count_fn, fill_fn, device, stream) -> SubspaceHandle:
    count = ctypes.c_uint64(0)
    _check(count_fn(ctypes.byref(count)))
    n = int(count.value)
    tiles = torch.empty((max(n, 1), 2), dtype=torch.int64, device=device)
    _check(fill_fn(tiles, n, ctypes.byref(count)))
    t = tiles[:n]
    numel = int((t[:, 1] - t[:, 0]).sum().item()) if n else 0
    return SubspaceHandle(SUBSPACE_TILES, t, numel)


def tiles_from_ranges(ranges, tile_size: int = DEFAULT_TILE, device="cuda", stream=None) -> SubspaceHandle:
    b = np.ascontiguousarray([r[0] for r in ranges], np.uint64)
    e = np.ascontiguousarray([r[1] for r in ranges], np.uint64)
    L, s = load(), _stream(stream)
    return _tiles_result(
        lambda cnt: L.copes_tiles_from_ranges(_np_ptr(b), _np_ptr(e), len(ranges), tile_size, None, 0, cnt, s),
        lambda t, n, cnt: L.copes_tiles_from_ranges(_np_ptr(b), _np_ptr(e), len(ranges), tile_size,
                                                    _ptr(t), n, cnt, s), device, stream)


def subspace_build(layout: Layout, mode: int, K: int, k: int, seed: int = 0, chunk: int = 65536,
                   group_of: Optional[Sequence[int]] = None, chunk_map: Optional[torch.Tensor] = None,
                   tile_size: int = DEFAULT_TILE, device="cuda", stream=None) -> SubspaceHandle:
    """copes_subspace_build for the range modes (CONTIGUOUS, TENSOR_GROUPS, RANDOM_CHUNKS)."""
    g = None if group_of is None else np.ascontiguousarray(group_of, np.int32)
    spec = PartitionSpec(mode, K, seed, chunk, _np_ptr(g))
    L, s = load(), _stream(stream)
    cm = _ptr(chunk_map)
    return _tiles_result(
        lambda cnt: L.copes_subspace_build(ctypes.byref(layout.desc), ctypes.byref(spec), k, tile_size,
                                           cm, None, 0, cnt, s),
        lambda t, n, cnt: L.copes_subspace_build(ctypes.byref(layout.desc), ctypes.byref(spec), k,
                                                 tile_size, cm, _ptr(t), n, cnt, s), device, stream)


def random_chunk_map(n_chunks: int, K: int, seed: int, device="cuda", stream=None) -> torch.Tensor:
    """copes_random_chunk_map with a torch-allocated sort workspace."""
    L = load()
    out = torch.empty(n_chunks, dtype=torch.int32, device=device)
    nbytes = L.copes_random_chunk_map_workspace_bytes(n_chunks)
    ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=device)
    _check(L.copes_random_chunk_map(n_chunks, K, seed, _ptr(out), _ptr(ws), nbytes, _stream(stream)))
    if stream is not None:
        ws.record_stream(stream)  # freed in stream order with the sort's kernels
    return out


def hash_partition(layout: Layout, K: int, seed: int, device="cuda", stream=None) -> List[SubspaceHandle]:
    """copes_hash_count + copes_hash_fill: K sorted int64 index lists (torch-allocated)."""
    L, s = load(), _stream(stream)
    nbytes = L.copes_hash_workspace_bytes(ctypes.byref(layout.desc), K)
    if nbytes == 0:
        raise CopesError(ERR_INVALID_ARG, "copes_hash_workspace_bytes rejected the layout / K")
    ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    counts = np.zeros(K, np.uint64)
    _check(L.copes_hash_count(ctypes.byref(layout.desc), K, seed, _ptr(ws), nbytes, _np_ptr(counts), s))
    lists = [torch.empty(max(int(c), 2), dtype=torch.int64, device=device) for c in counts]
    ptrs = (ctypes.c_void_p * K)(*[t.data_ptr() for t in lists])
    _check(L.copes_hash_fill(ctypes.byref(layout.desc), K, seed, _ptr(ws), nbytes, ptrs, s))
    if stream is not None:
        ws.record_stream(stream)  # freed in stream order with the fill's kernels
    return [SubspaceHandle(SUBSPACE_INDICES, t[:int(c)], int(c)) for t, c in zip(lists, counts)]


def hash_partition_static(layout: Layout, K: int, seed: int, device="cuda", stream=None) -> List[SubspaceHandle]:
    """copes_hash_partition_static: the same K sorted index lists as hash_partition, built
    on the library's fixed static scratch instead of a workspace (for callers that cannot
    allocate device scratch; the lists themselves are still allocated here by torch)."""
    L, s = load(), _stream(stream)
    counts = np.zeros(K, np.uint64)
    _check(L.copes_hash_partition_static(ctypes.byref(layout.desc), K, seed, None, None, _np_ptr(counts), s))
    lists = [torch.empty(max(int(c), 2), dtype=torch.int64, device=device) for c in counts]
    ptrs = (ctypes.c_void_p * K)(*[t.data_ptr() for t in lists])
    caps = np.array([t.numel() for t in lists], np.uint64)
    _check(L.copes_hash_partition_static(ctypes.byref(layout.desc), K, seed, ptrs, _np_ptr(caps),
                                         _np_ptr(counts), s))
    return [SubspaceHandle(SUBSPACE_INDICES, t[:int(c)], int(c)) for t, c in zip(lists, counts)]


def hash_replay_partition(layout: Layout, K: int, seed: int, count: bool = True, device="cuda",
                          stream=None) -> List[SubspaceHandle]:
    """copes_hash_replay_subspace for k = 0..K-1: the K subspaces of the hash partition
    (K, seed) as HASH_REPLAY subspaces sharing one device tensor table; no index list is
    built.  count=True also counts the members (copes_hash_count on a temporary workspace)
    so that each handle's numel is known; otherwise numel is -1."""
    L, s = load(), _stream(stream)
    nbytes = L.copes_hash_replay_bytes(ctypes.byref(layout.desc))
    if nbytes == 0:
        raise CopesError(ERR_INVALID_ARG, "copes_hash_replay_bytes rejected the layout")
    table = torch.empty(nbytes, dtype=torch.uint8, device=device)
    counts = np.full(K, -1, np.int64)
    if count:
        wbytes = L.copes_hash_workspace_bytes(ctypes.byref(layout.desc), K)
        ws = torch.empty(wbytes, dtype=torch.uint8, device=device)
        c = np.zeros(K, np.uint64)
        _check(L.copes_hash_count(ctypes.byref(layout.desc), K, seed, _ptr(ws), wbytes, _np_ptr(c), s))
        counts = c.astype(np.int64)
    handles = []
    for k in range(K):
        S = Subspace()
        _check(L.copes_hash_replay_subspace(ctypes.byref(layout.desc), K, seed, k, _ptr(table), nbytes, s,
                                            ctypes.byref(S)))
        handles.append(SubspaceHandle(SUBSPACE_HASH_REPLAY, table, int(counts[k]), S))
    return handles


# -------------------------------------------------------------------------- ES steps
def perturb(arena: Arena, sub: SubspaceHandle, seed: int, signed_sigma: float, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_perturb(ctypes.byref(arena.params), ctypes.byref(S), seed, signed_sigma, _stream(stream)))


def subspace_spans(arena: Arena, subs: Sequence[SubspaceHandle]) -> List[Tuple[int, int]]:
    """[lo, hi) global-index span of each subspace (lo rounded down to a multiple of 4, as
    partner buffers need), read from the device in one copy; (0, 0) for an empty one."""
    spans = []
    for sub in subs:
        if sub.kind == SUBSPACE_TILES and sub.tensor.shape[0]:
            spans.append(torch.stack([sub.tensor[:, 0].min(), sub.tensor[:, 1].max()]))
        elif sub.kind == SUBSPACE_INDICES and sub.tensor.numel():
            spans.append(torch.stack([sub.tensor[0], sub.tensor[-1] + 1]))
        elif sub.kind == SUBSPACE_HASH_REPLAY:
            spans.append(torch.tensor([0, arena.w.numel()], device=arena.w.device))
        else:
            spans.append(torch.zeros(2, dtype=torch.int64, device=arena.w.device))
    if not spans:
        return []
    s = torch.stack(spans).cpu().numpy()
    return [(int(lo) & ~3, int(hi)) if hi > lo else (0, 0) for lo, hi in s]


def partner_buffer(arena: Arena, subs: Sequence[SubspaceHandle]) -> Tuple[torch.Tensor, int]:
    """A partner buffer (working dtype) covering every element of `subs`, and its base
    global index."""
    spans = [x for x in subspace_spans(arena, subs) if x[1] > x[0]]
    lo = min((x[0] for x in spans), default=0)
    hi = max((x[1] for x in spans), default=0)
    return torch.empty(max(hi - lo, 8), dtype=arena.w.dtype, device=arena.w.device), lo


def _partner_view(arena, partner: torch.Tensor, base: int) -> torch.Tensor:
    assert partner.is_cuda and partner.dtype == arena.w.dtype and partner.is_contiguous()
    return partner[:max(0, min(partner.numel(), arena.w.numel() - base))]


def perturb_pair(arena: Arena, sub: SubspaceHandle, seed: int, signed_sigma: float, partner: torch.Tensor,
                 base: int = 0, stream=None) -> None:
    """copes_perturb_pair: w as perturb(signed_sigma) and the partner member's weights
    (-signed_sigma) into `partner` (element g at partner[g - base])."""
    view = _partner_view(arena, partner, base)
    S = sub.struct()
    _check(load().copes_perturb_pair(ctypes.byref(arena.params), ctypes.byref(S), seed, signed_sigma,
                                     _ptr(partner), base, view.numel(), _stream(stream)))


def perturb_two_pairs(arena: Arena, sub: SubspaceHandle, seed_a: int, seed_b: int, signed_sigma: float,
                      stream=None) -> None:
    """copes_perturb_two_pairs: w = perturb(seed_a, +s), w2 = perturb(seed_a, -s),
    w3 = perturb(seed_b, +s), w4 = perturb(seed_b, -s) in one pass (four working copies,
    TILES subspaces)."""
    S = sub.struct()
    _check(load().copes_perturb_two_pairs(ctypes.byref(arena.params), ctypes.byref(S), seed_a, seed_b,
                                          signed_sigma, _stream(stream)))


def perturb_partner(arena: Arena, sub: SubspaceHandle, partner: torch.Tensor, base: int = 0,
                    stream=None) -> None:
    """copes_perturb_partner: w[g] = partner[g - base] for g in the subspace."""
    view = _partner_view(arena, partner, base)
    S = sub.struct()
    _check(load().copes_perturb_partner(ctypes.byref(arena.params), ctypes.byref(S), _ptr(partner), base,
                                        view.numel(), _stream(stream)))


def restore(arena: Arena, sub: SubspaceHandle, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_restore(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))


def context_commit(arena: Arena, sub: SubspaceHandle, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_context_commit(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))


def gather_master(arena: Arena, sub: SubspaceHandle, stream=None) -> torch.Tensor:
    """Gives an INDICES subspace a gathered master (allocated here, n_index fp32) filled
    with master[index[p]]; the ES steps over `sub` then read and update that copy."""
    assert sub.kind == SUBSPACE_INDICES
    if sub.gathered is None:
        sub.gathered = torch.empty(max(sub.tensor.numel(), 1), dtype=torch.float32, device=sub.tensor.device)
    S = sub.struct()
    _check(load().copes_gather_master(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))
    return sub.gathered


def hash_replay_mask(arena: Arena, sub: SubspaceHandle, buffer: Optional[torch.Tensor] = None,
                     stream=None) -> torch.Tensor:
    """copes_hash_replay_mask: hashes every element once and stores the membership bits
    of the replay subspace `sub`; its ES steps then read them instead of hashing.  `buffer`
    (int32, n_replay_tiles * 512) may be shared by the subspaces visited one at a time."""
    assert sub.kind == SUBSPACE_HASH_REPLAY
    words = int(sub.replay.n_replay_tiles) * 512
    if buffer is None:
        buffer = torch.empty(words, dtype=torch.int32, device=sub.tensor.device)
    assert buffer.dtype == torch.int32 and buffer.numel() >= words
    sub.mask = buffer
    sub.replay.replay_mask = buffer.data_ptr()
    _check(load().copes_hash_replay_mask(ctypes.byref(arena.params), ctypes.byref(sub.replay), _stream(stream)))
    return buffer


def drop_replay_mask(sub: SubspaceHandle) -> None:
    """Back to hashing membership in every kernel."""
    sub.mask = None
    sub.replay.replay_mask = None


def scatter_master(arena: Arena, sub: SubspaceHandle, stream=None) -> None:
    """Writes the gathered copy back: master[index[p]] = gathered[p]."""
    S = sub.struct()
    _check(load().copes_scatter_master(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))


def init_normal(arena: Arena, sub: SubspaceHandle, seed: int, mean: float, scale: float, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_init_normal(ctypes.byref(arena.params), ctypes.byref(S), seed, mean, scale,
                                    _stream(stream)))


def shape_fitness(rewards: torch.Tensor, mode, group: Optional[torch.Tensor] = None,
                  out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    mode = SHAPE_MODES[mode] if isinstance(mode, str) else mode
    assert rewards.dtype == torch.float32 and rewards.is_cuda and rewards.is_contiguous()
    if out is None:
        out = torch.empty_like(rewards)
    _check(load().copes_shape_fitness(_ptr(rewards), rewards.numel(), _ptr(group), mode, _ptr(out),
                                      _stream(stream)))
    return out


def update(arena: Arena, sub: SubspaceHandle, noise_id: np.ndarray, sign: np.ndarray,
           fitness: torch.Tensor, seeds: np.ndarray, coef: float, fuse_commit: bool = True,
           stream=None) -> None:
    nid = np.ascontiguousarray(noise_id, np.int32)
    sg = np.ascontiguousarray(sign, np.int8)
    sd = np.ascontiguousarray(seeds, np.uint64)
    S = sub.struct()
    _check(load().copes_update(ctypes.byref(arena.params), ctypes.byref(S), nid.size, _np_ptr(nid),
                               _np_ptr(sg), _ptr(fitness), sd.size, _np_ptr(sd), coef,
                               int(fuse_commit), _stream(stream)))


# ----------------------------------------------------------------------------- debug
def debug_philox(seed: int, q0: int, n: int, aux: int = 0, tag: int = TAG_NOISE, stream=None) -> torch.Tensor:
    out = torch.empty(4 * n, dtype=torch.int32, device="cuda")
    _check(load().copes_debug_philox(seed, q0, n, aux, tag, _ptr(out), _stream(stream)))
    return out


def debug_normals(seed: int, g0: int, n: int, tag: int = TAG_NOISE, stream=None) -> torch.Tensor:
    out = torch.empty(n, dtype=torch.float32, device="cuda")
    _check(load().copes_debug_normals(seed, tag, g0, n, _ptr(out), _stream(stream)))
    return out


def debug_transform(words: torch.Tensor, stream=None) -> torch.Tensor:
    out = torch.empty(words.numel(), dtype=torch.float32, device=words.device)
    _check(load().copes_debug_transform(_ptr(words), words.numel(), _ptr(out), _stream(stream)))
    return out


# ------------------------------------------------------------------ CPU weight backup
class BackupArena:
    """CPU weight backup mode: bf16 working weights on the device and the shared context as
    a bf16 copy in page-locked host memory (no fp32 master)."""

    def __init__(self, w: torch.Tensor, backup: torch.Tensor):
        assert w.is_cuda and w.dtype == torch.bfloat16 and w.is_contiguous()
        assert backup.dtype == torch.bfloat16 and not backup.is_cuda and backup.numel() == w.numel()
        self.w, self.backup = w, backup
        self.live = w  # the working buffer holding the member being evaluated
        self.params = BackupParams(w.data_ptr(), backup.data_ptr(), w.numel())

    @classmethod
    def empty(cls, n: int, device="cuda"):
        return cls(torch.empty(n, dtype=torch.bfloat16, device=device),
                   torch.empty(n, dtype=torch.bfloat16).pin_memory())


def backup_save(arena: BackupArena, sub: SubspaceHandle, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_backup_save(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))


def backup_perturb(arena: BackupArena, sub: SubspaceHandle, seed: int, signed_sigma: float, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_backup_perturb(ctypes.byref(arena.params), ctypes.byref(S), seed, signed_sigma,
                                       _stream(stream)))


def backup_perturb_pair(arena: BackupArena, sub: SubspaceHandle, seed: int, signed_sigma: float,
                        partner: torch.Tensor, base: int = 0, stream=None) -> None:
    """copes_backup_perturb_pair: w as backup_perturb(signed_sigma), the partner member's
    weights (-signed_sigma) into the device buffer `partner` (element g at partner[g - base])."""
    view = _partner_view(arena, partner, base)
    S = sub.struct()
    _check(load().copes_backup_perturb_pair(ctypes.byref(arena.params), ctypes.byref(S), seed, signed_sigma,
                                            _ptr(partner), base, view.numel(), _stream(stream)))


def backup_perturb_partner(arena: BackupArena, sub: SubspaceHandle, partner: torch.Tensor, base: int = 0,
                           stream=None) -> None:
    """copes_backup_perturb_partner: w[g] = partner[g - base] for g in the subspace."""
    view = _partner_view(arena, partner, base)
    S = sub.struct()
    _check(load().copes_backup_perturb_partner(ctypes.byref(arena.params), ctypes.byref(S), _ptr(partner), base,
                                               view.numel(), _stream(stream)))


def backup_restore(arena: BackupArena, sub: SubspaceHandle, stream=None) -> None:
    S = sub.struct()
    _check(load().copes_backup_restore(ctypes.byref(arena.params), ctypes.byref(S), _stream(stream)))


def backup_update(arena: BackupArena, sub: SubspaceHandle, noise_id: np.ndarray, sign: np.ndarray,
                  fitness: torch.Tensor, seeds: np.ndarray, coef: float, stream=None) -> None:
    nid = np.ascontiguousarray(noise_id, np.int32)
    sg = np.ascontiguousarray(sign, np.int8)
    sd = np.ascontiguousarray(seeds, np.uint64)
    assert fitness.dtype == torch.float32 and fitness.is_cuda and fitness.numel() == nid.size
    S = sub.struct()
    _check(load().copes_backup_update(ctypes.byref(arena.params), ctypes.byref(S), nid.size, _np_ptr(nid),
                                      _np_ptr(sg), _ptr(fitness), sd.size, _np_ptr(sd), coef, _stream(stream)))
