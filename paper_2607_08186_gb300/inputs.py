"""Seeded synthetic inputs shared by the tests, the smoke check and the benchmark.

This module holds no attention or expansion arithmetic: it only draws random
tensors with a CPU ``torch.Generator`` so the CUDA path and the CPU oracle can
be fed identical bytes.  The shapes mirror the paper's workloads (Qwen3-8B-class
dense attention: Hq=32, Hkv=8, Dh=128; large-MoE-class: Hq=64, Hkv=8, Dh=128;
expansion factors n in {1, 2, 4, 8}); the paper's data and weights are not
available, so N(0, 1) activations and N(0, 0.02) embedding tables stand in.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

WITHIN, CROSS, LOCAL, WITHIN_NAIVE = 0, 1, 2, 3


@dataclass(frozen=True)
class AttnShape:
    B: int
    L: int        # tokens per sequence (before expansion)
    n: int        # expansion factor (streams per token)
    Hq: int
    Hkv: int
    Dh: int

    @property
    def nL(self) -> int:
        return self.n * self.L


# Named workloads (tokens L before expansion; the kernels see n*L positions).
SHAPES = {
    "tiny": AttnShape(1, 64, 2, 4, 4, 64),
    "qwen3_8b_n4": AttnShape(1, 4096, 4, 32, 8, 128),
    "moe_large_n4": AttnShape(1, 8192, 4, 64, 8, 128),
}


def _randn(shape, seed: int, std: float = 1.0) -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    out = torch.empty(shape, dtype=torch.bfloat16)
    flat = out.view(-1)
    chunk = 1 << 26
    for i in range(0, flat.numel(), chunk):
        x = torch.randn(min(chunk, flat.numel() - i), generator=g, dtype=torch.float32)
        if std != 1.0:
            x.mul_(std)
        flat[i:i + x.numel()] = x.to(torch.bfloat16)
    return out


def attn_inputs(s: AttnShape, seed: int = 0, with_grad: bool = True):
    """Q, K, V (and dO) in bf16, N(0, 1), layouts [B][nL][H][Dh].

    Seeds: seed+0 -> Q, seed+1 -> K, seed+2 -> V, seed+3 -> dO."""
    q = _randn((s.B, s.nL, s.Hq, s.Dh), seed)
    k = _randn((s.B, s.nL, s.Hkv, s.Dh), seed + 1)
    v = _randn((s.B, s.nL, s.Hkv, s.Dh), seed + 2)
    if not with_grad:
        return q, k, v
    do = _randn((s.B, s.nL, s.Hq, s.Dh), seed + 3)
    return q, k, v, do


def embed_inputs(B: int, L: int, n: int, V: int, D: int, seed: int = 0):
    """n embedding tables bf16 [n][V][D] ~ N(0, 0.02) and token ids int32 [B][L] ~ U[0, V)."""
    tables = _randn((n, V, D), seed, std=0.02)
    g = torch.Generator(device="cpu")
    g.manual_seed(seed + 1000)
    ids = torch.randint(0, V, (B, L), generator=g, dtype=torch.int64).to(torch.int32)
    return tables, ids


def normal_bf16(shape, seed: int, std: float = 1.0) -> torch.Tensor:
    """bf16 tensor ~ N(0, std^2) from a seeded CPU generator (gradients of the expanded rows)."""
    return _randn(tuple(shape), seed, std=std)


def token_ids(B: int, L: int, V: int, seed: int, zipf: float = 0.0) -> torch.Tensor:
    """Token ids int32 [B][L].  zipf = 0: U[0, V).  zipf = a > 0: P(id = r) proportional to
    (r + 1)^-a, the rank-frequency shape of natural-language tokens, so frequent ids repeat
    many times within a batch (ranks are taken as ids; no permutation)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(seed + 2000)
    if zipf <= 0.0:
        return torch.randint(0, V, (B, L), generator=g, dtype=torch.int64).to(torch.int32)
    w = torch.arange(1, V + 1, dtype=torch.float64).pow(-zipf)
    ids = torch.multinomial(w, B * L, replacement=True, generator=g)
    return ids.view(B, L).to(torch.int32)
