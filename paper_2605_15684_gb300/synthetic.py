"""Seeded synthetic inputs shaped like the paper's DiT attention workloads.

This module holds no arithmetic of the method: it only draws tensors. Both the
CUDA path and the CPU oracle are fed from it, so it imports neither.

Workload geometry (Sec. 2.2, first paragraph): an f8c16 VAE turns a P x P image
into a 16 x P/8 x P/8 latent, and 2 x 2 patchify leaves a (P/16) x (P/16) grid of
image tokens; 512 px -> 32 x 32 = 1024 tokens, 1024 px -> 64 x 64 = 4096,
2048 px -> 128 x 128 = 16384. Heads are 24 x 64 as in the 1024 px DiT.

Recipe: a CPU ``torch.Generator`` seeded with ``seed`` draws Q, K then V, each
i.i.d. N(0, 1) in fp32 with shape [B, heads, N, d], multiplied by ``std`` and
then cast to the requested dtype (bf16 rounding happens in that cast).
"""
from __future__ import annotations

from dataclasses import dataclass

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    heads: int
    H_tok: int
    W_tok: int
    head_dim: int
    rho: float
    dtype: torch.dtype
    std: float = 1.0

    @property
    def N(self) -> int:
        return self.H_tok * self.W_tok


def tokens_for_image(pixels: int) -> int:
    """Side of the image-token grid for a square image: /8 (VAE) then /2 (patchify)."""
    return pixels // 16


# Workloads of the paper's 512-2048 px settings (the 512 px one scales by 1/sqrt(64)).
TINY = Workload("tiny-16x16-h2-fp32", 1, 2, 16, 16, 64, 0.75, torch.float32)
PX512 = Workload("512px-32x32-h24-bf16", 1, 24, 32, 32, 64, 0.8416, torch.bfloat16, 0.125)
PX1024 = Workload("1024px-64x64-h24-bf16", 1, 24, 64, 64, 64, 0.8416, torch.bfloat16)
PX2048 = Workload("2048px-128x128-h24-bf16", 1, 24, 128, 128, 64, 0.84, torch.bfloat16)


def qkv(B: int, heads: int, N: int, d: int, dtype=torch.bfloat16, seed: int = 0,
        std: float = 1.0):
    """Q, K, V on the CPU, [B, heads, N, d], drawn in that order from one seeded stream."""
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    shape = (B, heads, N, d)
    out = []
    for _ in range(3):
        x = torch.randn(shape, generator=g, dtype=torch.float32)
        if std != 1.0:
            x = x * std
        out.append(x.to(dtype).contiguous())
    return tuple(out)


def workload_qkv(w: Workload, seed: int = 0):
    return qkv(w.B, w.heads, w.N, w.head_dim, w.dtype, seed, w.std)


def feature_map(N: int, C: int, H: int, W: int, dtype=torch.float32, seed: int = 0):
    """A VAE feature map on the CPU, [N, C, H, W], i.i.d. N(0, 1) drawn in fp32 from one seeded
    stream, then cast to ``dtype``."""
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return torch.randn((N, C, H, W), generator=g, dtype=torch.float32).to(dtype).contiguous()


def projection_inputs(B: int, N: int, Dm: int, seed: int = 0):
    """Image-token activations and a QKV projection, on the CPU, drawn in this order from one
    seeded stream: X [B, N, Dm] ~ N(0, 1) cast to bf16, Wqkv [3 Dm, Dm] ~ N(0, 1/Dm) cast to
    bf16 (so that every projected channel has unit variance), bias [3 Dm] ~ N(0, 0.1^2) fp32."""
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    X = torch.randn((B, N, Dm), generator=g, dtype=torch.float32).to(torch.bfloat16).contiguous()
    Wqkv = (torch.randn((3 * Dm, Dm), generator=g, dtype=torch.float32) / Dm ** 0.5).to(torch.bfloat16).contiguous()
    bias = (0.1 * torch.randn((3 * Dm,), generator=g, dtype=torch.float32)).contiguous()
    return X, Wqkv, bias
