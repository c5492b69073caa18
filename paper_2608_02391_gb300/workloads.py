"""Seeded synthetic workloads shared by the CUDA path's tests/benchmark and the oracle.

This module holds none of the method's arithmetic: it describes parameter layouts
(decoder-shaped tensor tables), subspace groupings, hyper-parameters and seeded reward
/ weight generators drawn with numpy's PCG64.  Both sides receive identical inputs from
here; noise, perturbation, shaping and updates are computed by each side on its own.

Sizes reproduce the parameter counts named for the ES workloads:
  tiny      1,048,576 fp32 parameters (one vector)
  0.5B      24 layers, hidden 896, MLP 4864, vocab 151936, 14 q / 2 kv heads of 64, qkv
            bias, tied embeddings                              -> 494,032,768
  4B        36 layers, hidden 2560, MLP 9728, vocab 151936, 32 q / 8 kv heads of 128,
            q/k norms, tied embeddings                         -> 4,022,468,096
  8B        36 layers, hidden 4096, MLP 12288, vocab 151936, 32 q / 8 kv heads of 128,
            q/k norms, untied lm_head                          -> 8,190,735,360
The paper trains Qwen3.5-4B (4,659,865,088 parameters, Supp. B); no weights are needed
here because the ES step never reads them as a model, only as a vector.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

ALIGN = 64  # tensor t+1 starts at the next multiple of 64 after tensor t


@dataclass(frozen=True)
class Tensor:
    name: str
    numel: int
    kind: str  # "embed" | "attn" | "mlp" | "norm" | "bias" | "lm_head" | "vector"
    layer: int = -1


def layout_offsets(tensors: Sequence[Tensor]) -> List[int]:
    off = [0]
    for t in tensors:
        off.append((off[-1] + t.numel + ALIGN - 1) // ALIGN * ALIGN)
    return off


def decoder_tensors(layers, hidden, mlp, vocab, q_heads, kv_heads, head_dim, qkv_bias,
                    qk_norm, tied) -> List[Tensor]:
    q_out, kv_out = q_heads * head_dim, kv_heads * head_dim
    ts = [Tensor("embed", vocab * hidden, "embed")]
    for l in range(layers):
        ts.append(Tensor(f"l{l}.q", hidden * q_out, "attn", l))
        if qkv_bias:
            ts.append(Tensor(f"l{l}.q_bias", q_out, "bias", l))
        ts.append(Tensor(f"l{l}.k", hidden * kv_out, "attn", l))
        if qkv_bias:
            ts.append(Tensor(f"l{l}.k_bias", kv_out, "bias", l))
        ts.append(Tensor(f"l{l}.v", hidden * kv_out, "attn", l))
        if qkv_bias:
            ts.append(Tensor(f"l{l}.v_bias", kv_out, "bias", l))
        ts.append(Tensor(f"l{l}.o", q_out * hidden, "attn", l))
        if qk_norm:
            ts.append(Tensor(f"l{l}.q_norm", head_dim, "norm", l))
            ts.append(Tensor(f"l{l}.k_norm", head_dim, "norm", l))
        ts.append(Tensor(f"l{l}.in_norm", hidden, "norm", l))
        ts.append(Tensor(f"l{l}.gate", hidden * mlp, "mlp", l))
        ts.append(Tensor(f"l{l}.up", hidden * mlp, "mlp", l))
        ts.append(Tensor(f"l{l}.down", mlp * hidden, "mlp", l))
        ts.append(Tensor(f"l{l}.post_norm", hidden, "norm", l))
    ts.append(Tensor("final_norm", hidden, "norm"))
    if not tied:
        ts.append(Tensor("lm_head", vocab * hidden, "lm_head"))
    return ts


def tiny_tensors() -> List[Tensor]:
    return [Tensor("theta", 1 << 20, "vector")]


def qwen_0p5b_tensors() -> List[Tensor]:
    return decoder_tensors(24, 896, 4864, 151936, 14, 2, 64, True, False, True)


def qwen_4b_tensors() -> List[Tensor]:
    return decoder_tensors(36, 2560, 9728, 151936, 32, 8, 128, False, True, True)


def qwen_8b_tensors() -> List[Tensor]:
    return decoder_tensors(36, 4096, 12288, 151936, 32, 8, 128, False, True, False)


# ------------------------------------------------------------------- subspace groupings
def group_layer_blocks(tensors: Sequence[Tensor], K: int, n_layers: int,
                       embed_alone: bool) -> List[int]:
    """Group id per tensor for layer-block subspaces.

    embed_alone=False (4B): K blocks of layers cut at floor(L k / K); the embedding joins
    block 0 and the final norm the last block.
    embed_alone=True (0.5B): group 0 = embedding + final norm; the layers are cut into
    K-1 blocks at floor(L k / (K-1)) and numbered 1..K-1."""
    nb = K - 1 if embed_alone else K
    cuts = [n_layers * k // nb for k in range(nb + 1)]

    def block(l):
        for b in range(nb):
            if cuts[b] <= l < cuts[b + 1]:
                return b
        raise ValueError(l)

    out = []
    for t in tensors:
        if t.layer >= 0:
            out.append(block(t.layer) + (1 if embed_alone else 0))
        elif t.kind == "embed":
            out.append(0)
        else:  # final norm
            out.append(0 if embed_alone else nb - 1)
    return out


def group_by_type(tensors: Sequence[Tensor]) -> List[int]:
    """8B grouping: 0 attention, 1 MLP, 2 norms + embeddings, 3 lm_head."""
    code = {"attn": 0, "bias": 0, "mlp": 1, "norm": 2, "embed": 2, "lm_head": 3}
    return [code[t.kind] for t in tensors]


# -------------------------------------------------------------------------------- config
@dataclass
class Workload:
    name: str
    tensors: List[Tensor]
    K: int
    mode: str  # "contiguous" | "groups" | "hash" | "random_chunks"
    n_members: int
    sigma: float
    alpha: float
    shaping: str  # "zscore" | "zscore_grouped" | "centered_rank" | "none"
    pairing: str = "antithetic"
    convention: str = "openai"  # step coefficient alpha / (N sigma); "paper": alpha / N
    dimension_aware: bool = False
    working_dtype: str = "bf16"
    cycles: int = 1
    group_of: Optional[List[int]] = None
    partition_seed: int = 1088
    chunk: int = 65536
    base_seed: int = 33  # the paper's ES training seed (Supp. A.5)
    reward: str = "bernoulli_mean"
    reward_draws: int = 16
    reward_p: tuple = (0.2, 0.6)
    data_seed: int = 33
    init_seed: int = 0
    init_scale: float = 0.02
    extra: dict = field(default_factory=dict)

    @property
    def numel(self) -> List[int]:
        return [t.numel for t in self.tensors]

    @property
    def d(self) -> int:
        return sum(self.numel)

    @property
    def d_pad(self) -> int:
        return layout_offsets(self.tensors)[-1]


def workload(name: str) -> Workload:
    """The five ES workloads (tiny, 0.5B, 4B layer blocks, 4B hash, 8B by type)."""
    if name == "tiny":
        return Workload("tiny", tiny_tensors(), K=4, mode="contiguous", n_members=8,
                        sigma=1e-3, alpha=5e-4, shaping="zscore", working_dtype="fp32",
                        cycles=3, reward="linear", data_seed=33)
    if name == "0.5b":
        ts = qwen_0p5b_tensors()
        return Workload("0.5b", ts, K=8, mode="groups", n_members=16, sigma=1e-3, alpha=5e-4,
                        shaping="centered_rank", group_of=group_layer_blocks(ts, 8, 24, True),
                        reward="bernoulli_fixed", reward_draws=8, reward_p=(0.4, 0.4),
                        data_seed=34)
    if name == "4b":
        ts = qwen_4b_tensors()
        return Workload("4b", ts, K=8, mode="groups", n_members=32, sigma=1e-3, alpha=5e-4,
                        shaping="zscore", group_of=group_layer_blocks(ts, 8, 36, False),
                        data_seed=35)
    if name == "4b-hash":
        ts = qwen_4b_tensors()
        return Workload("4b-hash", ts, K=16, mode="hash", n_members=64, sigma=1e-3,
                        alpha=5e-4, shaping="zscore", data_seed=36)
    if name == "8b":
        ts = qwen_8b_tensors()
        return Workload("8b", ts, K=4, mode="groups", n_members=128, sigma=5e-4, alpha=5e-4,
                        shaping="zscore", group_of=group_by_type(ts), cycles=10, data_seed=37)
    if name == "4b-slice":
        # profiling case: the 4B workload's step on 4 tensors of 2^26 parameters (1.6 GB
        # resident: larger than L2, small enough for multi-pass counter captures)
        ts = [Tensor(f"block{i}", 1 << 26, "attn", i) for i in range(4)]
        return Workload("4b-slice", ts, K=4, mode="groups", n_members=32, sigma=1e-3, alpha=5e-4,
                        shaping="zscore", group_of=[0, 1, 2, 3], data_seed=35)
    if name == "4b-slice-big":
        # traffic-capture case: two subspaces of 2^28 parameters (4 GB resident with two
        # working copies), large enough that a kernel's unflushed L2 write-back at its end
        # is a small fraction of its DRAM bytes
        ts = [Tensor(f"block{i}", 1 << 28, "attn", i) for i in range(2)]
        return Workload("4b-slice-big", ts, K=2, mode="groups", n_members=32, sigma=1e-3, alpha=5e-4,
                        shaping="zscore", group_of=[0, 1], data_seed=35)
    if name == "4b-hash-slice":
        # profiling case of the hash workload: the same K = 16 hash partition and N = 64 on
        # 4 tensors of 2^26 parameters (1.6 GB resident)
        ts = [Tensor(f"block{i}", 1 << 26, "attn", i) for i in range(4)]
        return Workload("4b-hash-slice", ts, K=16, mode="hash", n_members=64, sigma=1e-3, alpha=5e-4,
                        shaping="zscore", data_seed=36)
    raise KeyError(name)


# ------------------------------------------------------------------------------ rewards
def bernoulli_rewards(rng: np.random.Generator, n: int, draws: int, p_lo: float,
                      p_hi: float) -> np.ndarray:
    """Mean of `draws` Bernoulli(p_i) per member, p_i ~ U(p_lo, p_hi): multiples of
    1/draws in [0, 1], as fp32."""
    p = rng.uniform(p_lo, p_hi, size=n) if p_hi > p_lo else np.full(n, p_lo)
    hits = rng.binomial(draws, p)
    return (hits / draws).astype(np.float32)


def reward_stream(w: Workload, steps: int) -> np.ndarray:
    """Rewards for `steps` visits of a subspace, shape [steps, N] (seeded by data_seed)."""
    rng = np.random.Generator(np.random.PCG64(w.data_seed))
    out = np.zeros((steps, w.n_members), dtype=np.float32)
    lo, hi = w.reward_p
    for s in range(steps):
        out[s] = bernoulli_rewards(rng, w.n_members, w.reward_draws, lo, hi)
    return out


def tiny_theta_and_objective(n: int = 1 << 20, seed_theta: int = 0, seed_c: int = 1):
    """theta ~ N(0, 0.02^2) (fp32) and the linear objective's coefficient vector c ~ N(0, 1)
    (fp64) for the tiny workload, both from PCG64."""
    theta = (np.random.Generator(np.random.PCG64(seed_theta)).standard_normal(n) * 0.02)
    c = np.random.Generator(np.random.PCG64(seed_c)).standard_normal(n)
    return theta.astype(np.float32), c


def gaussian_vector(n: int, seed: int, scale: float = 1.0) -> np.ndarray:
    return (np.random.Generator(np.random.PCG64(seed)).standard_normal(n) * scale).astype(np.float32)
