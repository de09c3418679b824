"""Seeded synthetic inputs shaped like the paper's LLaMA-2-7B workloads (Sec. 4.1).

This module draws random numbers only: it holds none of the method's arithmetic, and both the
CUDA path's tests/bench and the CPU oracle take their inputs from here. The paper's real
checkpoints and datasets (LLaMA-2-7B, C4, RedPajama) are stood in for by these shapes:

* weights: Student-t with 4 degrees of freedom scaled to std 0.02, drawn as
  0.02/sqrt(2) * z / sqrt(chi2_4 / 4), chi2_4 = z1^2 + z2^2 + z3^2 + z4^2 (Var t_4 = 2);
  the tiny layer uses iid N(0, 0.02^2);
* activations: N(0, 1) with round(1% of the real channels) outlier channels (a seeded
  permutation) scaled by 20, rounded to bf16 (the tiny layer keeps fp32 N(0, 1)).
"""
from __future__ import annotations

import torch

HIDDEN = 4096
INTERMEDIATE = 11008
LAYERS = 32
# (name, out_features, in_features) of the seven linears of a LLaMA-2-7B decoder layer
PROJECTIONS = (
    ("q", HIDDEN, HIDDEN), ("k", HIDDEN, HIDDEN), ("v", HIDDEN, HIDDEN), ("o", HIDDEN, HIDDEN),
    ("gate", INTERMEDIATE, HIDDEN), ("up", INTERMEDIATE, HIDDEN), ("down", HIDDEN, INTERMEDIATE),
)


def _gen(seed: int, device="cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def student_t_weight(rows: int, cols: int, seed: int, device="cpu") -> torch.Tensor:
    """fp32 [rows][cols] Student-t(df=4) entries with std 0.02."""
    g = _gen(seed, device)
    z = torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32)
    chi2 = torch.zeros_like(z)
    for _ in range(4):
        chi2 += torch.randn(rows, cols, generator=g, device=device, dtype=torch.float32) ** 2
    return (0.02 / 2 ** 0.5) * z / torch.sqrt(chi2 / 4.0)


def outlier_activations(tokens: int, features: int, seed: int, device="cpu") -> torch.Tensor:
    """bf16 [tokens][features]: N(0,1), round(0.01*features) outlier channels scaled x20."""
    g = _gen(seed, device)
    x = torch.randn(tokens, features, generator=g, device=device, dtype=torch.float32)
    k = int(round(0.01 * features))
    idx = torch.randperm(features, generator=g, device=device)[:k]
    x[:, idx] *= 20.0
    return x.to(torch.bfloat16)


def tiny_layer():
    """The 256x256 layer: A ~ N(0, 0.02^2) fp32 (seed 0), x: 4 tokens x 256 fp32 N(0,1) drawn
    after A from the same generator."""
    g = _gen(0)
    A = 0.02 * torch.randn(256, 256, generator=g, dtype=torch.float32)
    x = torch.randn(4, 256, generator=g, dtype=torch.float32)
    return A, x


def weight_seed(kind: str, idx: int = 0, proj: int = 0) -> int:
    """Seeds of the synthetic weights: attention layer 2, MLP layers 3000+i, prefill 4000+i,
    linear stack 5000 + 7*layer + projection index (q,k,v,o,gate,up,down = 0..6)."""
    return {"attn": 2, "mlp": 3000 + idx, "prefill": 4000 + idx,
            "stack": 5000 + 7 * idx + proj}[kind]


def activation_seed(weight_seed_value: int, tokens: int) -> int:
    return 1_000_003 * (weight_seed_value + 1) + tokens


def random_matrix(rows: int, cols: int, seed: int, scale: float = 1.0, dtype=torch.float32):
    """Generic seeded N(0, scale^2) matrix for parity sweeps over odd and ragged shapes."""
    g = _gen(seed)
    return (scale * torch.randn(rows, cols, generator=g, dtype=torch.float32)).to(dtype)
