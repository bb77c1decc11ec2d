"""Seeded synthetic inputs shared by the CUDA path's tests/benchmark and the
oracle's tests.

This module holds random draws and workload shapes only; none of the method's
arithmetic (layout, masking, softmax, retention) lives here. Sizes that depend
on the layout (the augmented length T, retained count R) are passed in by the
caller.

The draws stand in for the paper's genomic workloads (1 kb segments of
GRCh38 / OpenGenome2 / MSL39 with Evo-2-7B-shaped heads, W ~ 1 kb, k = 100;
Sec. 4.1, Table "Full configuration"): nucleotide ids uniform over {A,C,G,T},
Q/K/V i.i.d. normal in bf16. The default seed is 42, the paper's training seed.
"""
from __future__ import annotations

import numpy as np
import torch

DEFAULT_SEED = 42


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def nucleotides(B: int, N: int, seed: int = DEFAULT_SEED, device="cpu") -> torch.Tensor:
    """uint8 [B, N], ids uniform over {0,1,2,3} = {A,C,G,T}."""
    g = _gen(seed, device)
    return torch.randint(0, 4, (B, N), generator=g, device=device, dtype=torch.int64).to(torch.uint8)


def k_schedule(M: int, choices, seed: int = DEFAULT_SEED) -> np.ndarray:
    """int32 [M]: one cadence per window drawn uniformly from ``choices``
    (the randomized compression schedule of App. A.1, "slightly perturbing k")."""
    choices = np.asarray(list(choices), dtype=np.int32)
    if choices.size == 1:
        return np.full(M, choices[0], dtype=np.int32)
    rng = np.random.default_rng(seed)
    return choices[rng.integers(0, choices.size, size=M)].astype(np.int32)


def normal_bf16(shape, std: float, seed: int, device="cpu") -> torch.Tensor:
    """bf16 tensor of i.i.d. N(0, std^2) draws (drawn in fp32, rounded once)."""
    g = _gen(seed, device)
    x = torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16)


def qkv(shape, std: float = 1.0, seed: int = DEFAULT_SEED, device="cpu", q_per_kv: int = 1):
    """Three independent bf16 tensors (Q, K, V) of the given shape [B, H, ...];
    with q_per_kv = g > 1 (grouped-query heads) K and V have H / g heads."""
    kv_shape = tuple(shape) if q_per_kv <= 1 else (shape[0], shape[1] // q_per_kv) + tuple(shape[2:])
    return tuple(normal_bf16(shape if i == 0 else kv_shape, std, seed * 3 + i + 1, device) for i in range(3))


def start_fill(B: int, hi: int, seed: int = DEFAULT_SEED) -> np.ndarray:
    """int32 [B]: per-sequence current-window fill, uniform over {0..hi}."""
    rng = np.random.default_rng(seed + 7)
    return rng.integers(0, hi + 1, size=B).astype(np.int32)
