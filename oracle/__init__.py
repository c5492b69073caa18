"""CPU oracle for the CoPES evolution-strategy core (test infrastructure only).

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg may
import this package.  The product path -- the CUDA library in ``paper_2608_02391_gb300`` --
never imports it, and the two share no code.

The arithmetic lives in ``copes_oracle.c`` (plain C, fp64, one element at a time); this
module compiles it with gcc on first use and wraps it with ctypes/numpy.  Each wrapper
names the paper passage its C function follows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "copes_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

TAG_NOISE, TAG_INIT, TAG_PARTITION, TAG_SEED, TAG_CHUNK = 0, 1, 2, 3, 4
BF16, FP32 = 0, 1
SHAPE_NONE, SHAPE_ZSCORE, SHAPE_ZSCORE_GROUPED, SHAPE_CENTERED_RANK = 0, 1, 2, 3
ONE_SIDED, ANTITHETIC = 0, 1
COEF_PAPER, COEF_OPENAI = 0, 1

# Strict IEEE evaluation: no FMA contraction (gcc contracts by default on aarch64), no
# fast-math, so x86 and Arm hosts give the same fp64 arithmetic up to libm's last bit.
CFLAGS = ["-O2", "-std=gnu11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` next to the source if it is missing or stale."""
    with _lock:
        stale = (not os.path.exists(_LIB_PATH)
                 or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
        if force or stale:
            tmp = _LIB_PATH + f".tmp{os.getpid()}"
            subprocess.check_call(["gcc", *CFLAGS, _SRC, "-lm", "-o", tmp])
            os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class Subspace(ctypes.Structure):
    _fields_ = [
        ("kind", ctypes.c_int),
        ("n_ranges", ctypes.c_int),
        ("begin", ctypes.c_void_p),
        ("end", ctypes.c_void_p),
        ("idx", ctypes.c_void_p),
        ("n_idx", ctypes.c_uint64),
    ]


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        u64, u32, i32, dbl, flt, vp = (ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int,
                                       ctypes.c_double, ctypes.c_float, ctypes.c_void_p)
        sig = {
            "oracle_fault_flag": (i32, []),
            "oracle_clear_fault": (None, []),
            "oracle_philox4x32_10": (None, [vp, vp, vp]),
            "oracle_philox_stream": (None, [u64, u64, u64, u32, u32, vp]),
            "oracle_uniform": (dbl, [u32]),
            "oracle_normal_quantile": (dbl, [dbl]),
            "oracle_normal_quantile_array": (None, [vp, u64, vp]),
            "oracle_noise_at": (dbl, [u64, u32, u64]),
            "oracle_noise": (None, [u64, u32, vp, u64, vp]),
            "oracle_noise_range": (None, [u64, u32, u64, u64, vp]),
            "oracle_bf16_bits": (ctypes.c_uint16, [dbl]),
            "oracle_bf16_value": (dbl, [ctypes.c_uint16]),
            "oracle_perturb": (None, [vp, i32, vp, ctypes.POINTER(Subspace), u64, flt]),
            "oracle_perturb_at": (None, [u64, vp, vp, u64, flt, i32, vp, vp]),
            "oracle_restore": (None, [vp, i32, vp, ctypes.POINTER(Subspace)]),
            "oracle_commit": (None, [vp, i32, vp, ctypes.POINTER(Subspace)]),
            "oracle_shape_fitness": (i32, [vp, i32, vp, i32, vp]),
            "oracle_member_table": (i32, [i32, i32, vp, vp]),
            "oracle_member_seed": (u64, [u64, u32, u32, u32]),
            "oracle_sigma_eff": (dbl, [dbl, dbl, dbl, i32]),
            "oracle_step_coef": (dbl, [dbl, i32, dbl, i32]),
            "oracle_noise_weights": (None, [i32, vp, vp, vp, i32, vp]),
            "oracle_update_at": (None, [u64, vp, vp, i32, vp, vp, flt, vp, vp, vp]),
            "oracle_update": (i32, [vp, vp, i32, ctypes.POINTER(Subspace), i32, vp, vp, vp,
                                    i32, vp, flt]),
            "oracle_layout": (None, [vp, i32, vp]),
            "oracle_contiguous_ranges": (i32, [vp, vp, i32, i32, i32, vp, vp, i32]),
            "oracle_group_ranges": (i32, [vp, vp, i32, vp, i32, vp, vp, i32]),
            "oracle_hash_subspace": (u32, [u64, u32, u64, u32]),
            "oracle_hash_list": (u64, [vp, vp, vp, i32, u32, u64, u32, vp]),
            "oracle_random_chunks": (i32, [u64, u32, u64, vp]),
            "oracle_chunk_ranges": (i32, [vp, vp, i32, u64, vp, u32, vp, vp, i32]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def fault_flag() -> int:
    return lib().oracle_fault_flag()


def clear_fault() -> None:
    lib().oracle_clear_fault()


# ----------------------------------------------------------------------------- generator
def philox4x32_10(ctr, key):
    """One Philox4x32-10 block (SC'11): 4 counter words, 2 key words -> 4 words."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_philox4x32_10(_p(c), _p(k), _p(out))
    return out


def philox_stream(seed: int, q0: int, n: int, aux: int = 0, tag: int = TAG_NOISE):
    """Words for counters q0..q0+n-1 under this project's counter layout, shape [n, 4]."""
    out = np.zeros((n, 4), dtype=np.uint32)
    lib().oracle_philox_stream(seed, q0, n, aux, tag, _p(out))
    return out


def uniform(x: int) -> float:
    return lib().oracle_uniform(int(x))


def normal_quantile(u: float) -> float:
    return lib().oracle_normal_quantile(float(u))


def normal_quantile_array(u):
    """Phi^-1 elementwise over an fp64 array (values strictly inside (0, 1))."""
    u = np.ascontiguousarray(u, dtype=np.float64)
    out = np.zeros_like(u)
    lib().oracle_normal_quantile_array(_p(u), u.size, _p(out))
    return out


def noise(seed: int, g, tag: int = TAG_NOISE):
    """eps_seed[g] (fp64) for an array of global indices (Eq. 3 / Eq. 8 directions)."""
    g = np.ascontiguousarray(g, dtype=np.uint64)
    out = np.zeros(g.shape, dtype=np.float64)
    lib().oracle_noise(seed, tag, _p(g), g.size, _p(out))
    return out


def noise_range(seed: int, g0: int, n: int, tag: int = TAG_NOISE):
    out = np.zeros(n, dtype=np.float64)
    lib().oracle_noise_range(seed, tag, g0, n, _p(out))
    return out


# ------------------------------------------------------------------------------ rounding
def bf16_bits(x: float) -> int:
    return int(lib().oracle_bf16_bits(float(x)))


def bf16_bits_array(x):
    x = np.asarray(x, dtype=np.float64).ravel()
    f = lib().oracle_bf16_bits
    return np.array([f(float(v)) for v in x], dtype=np.uint16)


def bf16_value(bits: int) -> float:
    return lib().oracle_bf16_value(int(bits))


# ----------------------------------------------------------------------------- subspaces
def make_subspace(ranges=None, indices=None):
    """Subspace descriptor: a list of (begin, end) global ranges or an int64 index list.
    The returned tuple keeps the backing arrays alive."""
    if ranges is not None:
        b = np.ascontiguousarray([r[0] for r in ranges], dtype=np.uint64)
        e = np.ascontiguousarray([r[1] for r in ranges], dtype=np.uint64)
        s = Subspace(0, len(ranges), _p(b), _p(e), None, 0)
        return (s, b, e)
    idx = np.ascontiguousarray(indices, dtype=np.int64)
    s = Subspace(1, 0, None, None, _p(idx), idx.size)
    return (s, idx)


def _sref(sub):
    return ctypes.byref(sub[0])


def _dtype_code(w):
    if w.dtype == np.uint16:
        return BF16
    if w.dtype == np.float32:
        return FP32
    raise TypeError("working tensor must be uint16 (bf16 bits) or float32")


# ------------------------------------------------------------------------------ ES steps
def perturb(w, master, sub, seed: int, signed_sigma: float):
    """Eq. 8: w[g] = round(theta[g] + s sigma_k eps[g]) for g in S (in place)."""
    lib().oracle_perturb(_p(w), _dtype_code(w), _p(master), _sref(sub), seed,
                         np.float32(signed_sigma))


def perturb_at(g, theta, seed: int, signed_sigma: float, dtype: int):
    g = np.ascontiguousarray(g, dtype=np.uint64)
    theta = np.ascontiguousarray(theta, dtype=np.float32)
    bits = np.zeros(g.size, dtype=np.uint32)
    exact = np.zeros(g.size, dtype=np.float64)
    lib().oracle_perturb_at(g.size, _p(g), _p(theta), seed, np.float32(signed_sigma), dtype,
                            _p(bits), _p(exact))
    return bits, exact


def restore(w, master, sub):
    """Supp. A.8 direct restore: w[g] = round(theta[g]) for g in S (in place)."""
    lib().oracle_restore(_p(w), _dtype_code(w), _p(master), _sref(sub))


def commit(w, master, sub):
    """Context commit after the update: w[g] = round(theta+[g]) for g in S."""
    lib().oracle_commit(_p(w), _dtype_code(w), _p(master), _sref(sub))


def shape_fitness(r, mode: int, group=None):
    """Eq. 5 / Eq. 12 z-score, the Sec. 4.4 per-group variant, or centred ranks."""
    r = np.ascontiguousarray(r, dtype=np.float32)
    f = np.zeros_like(r)
    gp = None if group is None else np.ascontiguousarray(group, dtype=np.int32)
    rc = lib().oracle_shape_fitness(_p(r), r.size, _p(gp), mode, _p(f))
    if rc != 0:
        raise ValueError("oracle_shape_fitness rejected its arguments")
    return f


def member_table(n_members: int, pairing: int):
    noise_id = np.zeros(n_members, dtype=np.int32)
    sign = np.zeros(n_members, dtype=np.int8)
    n_noise = lib().oracle_member_table(n_members, pairing, _p(noise_id), _p(sign))
    if n_noise < 0:
        raise ValueError("antithetic pairing needs an even member count")
    return noise_id, sign, n_noise


def member_seed(base_seed: int, iteration: int, k: int, j: int) -> int:
    return int(lib().oracle_member_seed(base_seed, iteration, k, j))


def sigma_eff(sigma: float, d: float, d_k: float, dimension_aware: bool = True) -> float:
    """Eq. 11: sigma_k = sigma sqrt(d / d_k)."""
    return lib().oracle_sigma_eff(sigma, float(d), float(d_k), int(dimension_aware))


def step_coef(alpha: float, n_members: int, sigma_eff_: float, convention: int) -> float:
    return lib().oracle_step_coef(alpha, n_members, sigma_eff_, convention)


def noise_weights(noise_id, sign, f, n_noise: int):
    noise_id = np.ascontiguousarray(noise_id, dtype=np.int32)
    sign = np.ascontiguousarray(sign, dtype=np.int8)
    f = np.ascontiguousarray(f, dtype=np.float32)
    wj = np.zeros(n_noise, dtype=np.float64)
    lib().oracle_noise_weights(noise_id.size, _p(noise_id), _p(sign), _p(f), n_noise, _p(wj))
    return wj


def update_at(g, theta, seeds, wj, coef: float):
    """Eq. 13 at sampled indices: (rounded fp32 result, exact fp64 value, error scale)."""
    g = np.ascontiguousarray(g, dtype=np.uint64)
    theta = np.ascontiguousarray(theta, dtype=np.float32)
    seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
    wj = np.ascontiguousarray(wj, dtype=np.float64)
    out = np.zeros(g.size, dtype=np.float32)
    exact = np.zeros(g.size, dtype=np.float64)
    scale = np.zeros(g.size, dtype=np.float64)
    lib().oracle_update_at(g.size, _p(g), _p(theta), seeds.size, _p(seeds), _p(wj),
                           np.float32(coef), _p(out), _p(exact), _p(scale))
    return out, exact, scale


def update(master, sub, noise_id, sign, f, seeds, coef: float, w=None):
    """Eq. 13 over S, in place on master; with w given, the context commit follows."""
    noise_id = np.ascontiguousarray(noise_id, dtype=np.int32)
    sign = np.ascontiguousarray(sign, dtype=np.int8)
    f = np.ascontiguousarray(f, dtype=np.float32)
    seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
    dt = BF16 if w is None else _dtype_code(w)
    rc = lib().oracle_update(_p(master), _p(w), dt, _sref(sub), noise_id.size, _p(noise_id),
                             _p(sign), _p(f), seeds.size, _p(seeds), np.float32(coef))
    if rc != 0:
        raise MemoryError("oracle_update")


# ----------------------------------------------------------------------- layout / builds
def layout(numel):
    numel = np.ascontiguousarray(numel, dtype=np.uint64)
    off = np.zeros(numel.size + 1, dtype=np.uint64)
    lib().oracle_layout(_p(numel), numel.size, _p(off))
    return off


def _ranges_out(fn, *args, max_ranges=1 << 16):
    b = np.zeros(max_ranges, dtype=np.uint64)
    e = np.zeros(max_ranges, dtype=np.uint64)
    n = fn(*args, _p(b), _p(e), max_ranges)
    if n < 0:
        raise ValueError("too many ranges")
    return [(int(b[i]), int(e[i])) for i in range(n)]


def contiguous_ranges(numel, K: int, k: int):
    numel = np.ascontiguousarray(numel, dtype=np.uint64)
    off = layout(numel)
    return _ranges_out(lib().oracle_contiguous_ranges, _p(off), _p(numel), numel.size, K, k)


def group_ranges(numel, group_of, k: int):
    numel = np.ascontiguousarray(numel, dtype=np.uint64)
    group_of = np.ascontiguousarray(group_of, dtype=np.int32)
    off = layout(numel)
    return _ranges_out(lib().oracle_group_ranges, _p(off), _p(numel), numel.size, _p(group_of), k)


def hash_subspace(seed: int, tensor_id: int, e: int, K: int) -> int:
    return int(lib().oracle_hash_subspace(seed, tensor_id, e, K))


def hash_list(numel, tensor_ids, K: int, seed: int, k: int):
    numel = np.ascontiguousarray(numel, dtype=np.uint64)
    tids = np.ascontiguousarray(tensor_ids, dtype=np.uint32)
    off = layout(numel)
    n = lib().oracle_hash_list(_p(off), _p(numel), _p(tids), numel.size, K, seed, k, None)
    out = np.zeros(n, dtype=np.int64)
    lib().oracle_hash_list(_p(off), _p(numel), _p(tids), numel.size, K, seed, k, _p(out))
    return out


def random_chunks(n_chunks: int, K: int, seed: int):
    out = np.zeros(n_chunks, dtype=np.uint32)
    if lib().oracle_random_chunks(n_chunks, K, seed, _p(out)) != 0:
        raise MemoryError("oracle_random_chunks")
    return out


def chunk_ranges(numel, chunk: int, chunk_subspace, k: int):
    numel = np.ascontiguousarray(numel, dtype=np.uint64)
    cs = np.ascontiguousarray(chunk_subspace, dtype=np.uint32)
    off = layout(numel)
    return _ranges_out(lib().oracle_chunk_ranges, _p(off), _p(numel), numel.size, chunk, _p(cs), k)
