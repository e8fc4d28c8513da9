"""Seeded synthetic LLM-shaped inputs for the MixFP4 W4A4 linear layer.

This module generates inputs only: it holds none of the quantizer's or the
GEMM's arithmetic, so both the CUDA path and the CPU oracle can be fed from it.

The paper evaluates on Llama-3.1-8B / Qwen3 activations and weights (Sec. 4);
no checkpoints or datasets are used here.  Synthetic tensors with the same
shapes and the same qualitative statistics stand in for them:

* activations: Student-t with 3 degrees of freedom times 0.5, drawn as
  z0 / sqrt((z1^2 + z2^2 + z3^2) / 3) from standard normals, with 1 % of the
  K-channels (floor(0.01 K), chosen by a seeded permutation) scaled by 50 --
  the heavy-tailed, outlier-channel activations that motivate per-block
  format choice (Sec. 2.2, Fig. 2-3);
* weights: N(0, sigma), optionally times a per-output-row lognormal(0, 0.5)
  factor;
* the Hadamard-rotated case multiplies every 128-element chunk of a row by the
  normalised 128-point Walsh-Hadamard matrix (computed in float64), the
  orthogonal mixing the paper applies before quantization (Sec. 4, "+RHT").

Everything is drawn in fp32 on the CPU from ``torch.Generator`` seeds and cast
to bf16 with round-to-nearest-even.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def student_t3(rows: int, K: int, seed: int, scale: float = 0.5) -> torch.Tensor:
    """fp32 [rows, K] Student-t(df=3) * scale, generated row-chunk by row-chunk."""
    g = _gen(seed)
    out = torch.empty(rows, K, dtype=torch.float32)
    step = max(1, (1 << 24) // max(K, 1))
    for r0 in range(0, rows, step):
        r1 = min(rows, r0 + step)
        z = torch.randn(4, r1 - r0, K, generator=g, dtype=torch.float32)
        out[r0:r1] = z[0] / torch.sqrt((z[1] * z[1] + z[2] * z[2] + z[3] * z[3]) / 3.0) * scale
    return out


def outlier_channels(K: int, seed: int) -> torch.Tensor:
    n = int(math.floor(0.01 * K))
    return torch.randperm(K, generator=_gen(seed))[:n]


def activations(rows: int, K: int, seed: int, outlier_seed: int | None,
                outlier_gain: float = 50.0) -> torch.Tensor:
    x = student_t3(rows, K, seed)
    if outlier_seed is not None:
        x[:, outlier_channels(K, outlier_seed)] *= outlier_gain
    return x.to(torch.bfloat16)


def weights(N: int, K: int, seed: int, std: float, row_lognormal_sigma: float | None = None,
            outlier_seed: int | None = None, outlier_gain: float = 50.0) -> torch.Tensor:
    g = _gen(seed)
    w = torch.randn(N, K, generator=g, dtype=torch.float32) * std
    if row_lognormal_sigma is not None:
        w *= torch.exp(torch.randn(N, 1, generator=g, dtype=torch.float32) * row_lognormal_sigma)
    if outlier_seed is not None:
        w[:, outlier_channels(K, outlier_seed)] *= outlier_gain
    return w.to(torch.bfloat16)


def hadamard128(x: torch.Tensor) -> torch.Tensor:
    """Each row's 128-element chunks <- H_128 c / sqrt(128) (Sylvester order), fp64 -> bf16."""
    rows, K = x.shape
    assert K % 128 == 0
    h = torch.ones(1, 1, dtype=torch.float64)
    while h.shape[0] < 128:
        h = torch.cat([torch.cat([h, h], 1), torch.cat([h, -h], 1)], 0)
    h = h / math.sqrt(128.0)
    out = torch.empty(rows, K, dtype=torch.bfloat16)
    step = max(1, (1 << 22) // K)
    for r0 in range(0, rows, step):
        r1 = min(rows, r0 + step)
        c = x[r0:r1].to(torch.float64).reshape(r1 - r0, K // 128, 128)
        out[r0:r1] = (c @ h.T).reshape(r1 - r0, K).to(torch.bfloat16)
    return out


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 CPU tensor (what the oracle consumes)."""
    return t.contiguous().view(torch.int16).numpy().view("uint16")


@dataclass
class Linear:
    """One W4A4 linear: X [M, K] activations times W [N, K] weights."""
    name: str
    M: int
    N: int
    K: int
    x_seed: int
    w_seed: int
    outlier_seed: int | None
    w_std: float
    w_row_lognormal: float | None = None
    w_outliers: bool = False
    hadamard: bool = False

    def make_x(self) -> torch.Tensor:
        x = activations(self.M, self.K, self.x_seed, self.outlier_seed)
        return hadamard128(x) if self.hadamard else x

    def make_w(self) -> torch.Tensor:
        w = weights(self.N, self.K, self.w_seed, self.w_std, self.w_row_lognormal,
                    self.outlier_seed if self.w_outliers else None)
        return hadamard128(w) if self.hadamard else w


@dataclass
class Workload:
    name: str
    linears: list = field(default_factory=list)
    weights_prequantized: bool = True


def workloads() -> dict:
    """The five workloads, seeds X 1000+i, W 2000+i, outlier channels 3000+i (i = 1..5)."""
    w = {}
    w["tiny"] = Workload("tiny 128x512 . 256x512", [
        Linear("tiny", 128, 256, 512, 1001, 2001, None, 0.02)])
    w["attn"] = Workload("Llama-3-8B attention projection 2048x4096 . 4096x4096", [
        Linear("attn_proj", 2048, 4096, 4096, 1002, 2002, 3002, 0.02, w_row_lognormal=0.5)])
    w["mlp"] = Workload("Llama-3-8B MLP 4096x4096 -> 14336 (gate, up) -> 4096 (down)", [
        Linear("gate", 4096, 14336, 4096, 1003, 2003, 3003, 0.02, w_row_lognormal=0.5),
        Linear("up", 4096, 14336, 4096, 1003, 2103, 3003, 0.02, w_row_lognormal=0.5),
        Linear("down", 4096, 4096, 14336, 1103, 2203, 3103, 0.02, w_row_lognormal=0.5)])
    w["decode"] = Workload("decode 16x8192 . 28672x8192", [
        Linear("decode", 16, 28672, 8192, 1004, 2004, 3004, 0.015)])
    w["hadamard"] = Workload("Hadamard-rotated 8192x8192 . 8192x8192", [
        Linear("had", 8192, 8192, 8192, 1005, 2005, 3005, 0.02, w_outliers=True, hadamard=True)])
    return w


def sweep_activation(log2_elems: int, seed: int = 1006) -> torch.Tensor:
    """Quantizer-only sweep point: the attention activation distribution as [2^k / 4096, 4096]."""
    rows = (1 << log2_elems) // 4096
    return activations(rows, 4096, seed + log2_elems, 3006)
