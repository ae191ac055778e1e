"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module holds no step of the attention method: it only draws Q, K, V the way the
benchmark workloads are defined. Each tensor is i.i.d. N(0, 1) in fp32 from a seeded
torch generator; with ``outliers`` a seeded choice of max(1, round(0.01 * H * D))
channels of the flattened [H * D] axis is scaled by 8 (activation outlier channels of
Qwen2-class models); the result is rounded to the requested dtype (bf16: round to
nearest even). The draw happens on ``device``; CPU and CUDA generators give different
numbers for one seed, so a test draws once and copies the tensors to the other side.
"""
from __future__ import annotations

import torch


def outlier_count(H: int, D: int) -> int:
    return max(1, int(round(0.01 * H * D)))


def make_tensor(N: int, H: int, D: int, gen: torch.Generator, dtype=torch.bfloat16,
                outliers: bool = False, device="cpu") -> torch.Tensor:
    x = torch.randn(N, H * D, generator=gen, device=device, dtype=torch.float32)
    if outliers:
        n_out = outlier_count(H, D)
        idx = torch.randperm(H * D, generator=gen, device=device)[:n_out]
        x[:, idx] *= 8.0
    return x.view(N, H, D).to(dtype)


def make_qkv(N: int, Hq: int, Hkv: int, D: int, dtype=torch.bfloat16, seed: int = 0,
             outliers: bool = False, device="cpu"):
    """(q [N, Hq, D], k [N, Hkv, D], v [N, Hkv, D]) drawn from one generator seeded with ``seed``."""
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    q = make_tensor(N, Hq, D, gen, dtype, outliers, device)
    k = make_tensor(N, Hkv, D, gen, dtype, outliers, device)
    v = make_tensor(N, Hkv, D, gen, dtype, outliers, device)
    return q, k, v


def mask_seeds(n_seeds: int) -> list:
    """Ensemble seed values 0 .. n_seeds - 1."""
    return list(range(int(n_seeds)))
