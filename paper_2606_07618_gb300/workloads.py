"""Seeded synthetic inputs shaped like the paper's quantised tensors.

This module only draws random tensors; it holds none of the quantisation
arithmetic and is shared by the tests, the CPU oracle's callers and bench.py.
The paper's models and calibration data are not available, so each workload
is a stand-in with the shapes and value distributions stated below (all drawn
in float32 with a CPU ``torch.Generator`` and rounded to bf16 with RNE):

  weight-2048   one 2048x2048 matrix, N(0, 0.02^2), seed 0.
  llama8b       one Llama-3-8B layer: q/o 4096x4096, k/v 1024x4096,
                gate/up 14336x4096, down 4096x14336; N(0, 0.02^2) with
                round(0.001*in) input channels (columns) scaled x20; WMSE
                weights per input channel drawn lognormal(0, 1).
  act-8192      8192 tokens x 4096 hidden, Student-t(3) = z / sqrt(chi2_3/3)
                with 16 fixed channels x50 (per-call amax).
  kvq           K, V [16*8*4096, 128] and Q [16*32*4096, 128]: N(0, 1) times a
                per-head factor exp(0.5 * N(0, 1)) broadcast over batch, seq, dim.
  qwen72b       8192x29568 and 29568x8192, Laplace(0, 0.015) via
                -b*sgn(u)*ln(1-2|u|), round(0.0005*in) outlier columns x30,
                lognormal(0, 1) channel weights.
  table7-<B>    [B, 8192] activations with the act-8192 distribution (the
                batch sweep of the latency table in Appendix E).
Seeds: weight-2048 uses 0, others 1000*config_index + tensor_index.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


@dataclass
class Tensor:
    name: str
    rows: int
    cols: int
    dist: str                  # normal | student_t | kvq | laplace
    seed: int
    std: float = 0.02
    outlier_frac: float = 0.0
    outlier_count: int | None = None
    outlier_mult: float = 1.0
    heads: int = 0             # kvq: number of heads (rows = heads * per_head)
    weights: bool = False      # draw lognormal per-column weights for WMSE

    @property
    def numel(self) -> int:
        return self.rows * self.cols


@dataclass
class Workload:
    name: str
    tensors: list[Tensor]
    block: int = 16
    objective: str = "mse"     # mse | wmse
    fp8_div: float = 256.0     # D in S = amax / (6 D)
    dynamic_scale: bool = False
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def numel(self) -> int:
        return sum(t.numel for t in self.tensors)


def _llama8b() -> Workload:
    shapes = [("q", 4096, 4096), ("k", 1024, 4096), ("v", 1024, 4096), ("o", 4096, 4096),
              ("gate", 14336, 4096), ("up", 14336, 4096), ("down", 4096, 14336)]
    ts = [Tensor(n, r, c, "normal", 1000 * 1 + i, std=0.02, outlier_frac=0.001, outlier_mult=20.0, weights=True)
          for i, (n, r, c) in enumerate(shapes)]
    return Workload("llama8b", ts, block=16, objective="wmse", fp8_div=256.0)


def _kvq() -> Workload:
    ts = [Tensor("k", 16 * 8 * 4096, 128, "kvq", 3000, heads=8),
          Tensor("v", 16 * 8 * 4096, 128, "kvq", 3001, heads=8),
          Tensor("q", 16 * 32 * 4096, 128, "kvq", 3002, heads=32)]
    return Workload("kvq", ts, block=16, objective="mse", fp8_div=256.0)


def _qwen72b(block: int, objective: str) -> Workload:
    ts = [Tensor("w_8192x29568", 8192, 29568, "laplace", 4000, std=0.015, outlier_frac=0.0005, outlier_mult=30.0,
                 weights=True),
          Tensor("w_29568x8192", 29568, 8192, "laplace", 4001, std=0.015, outlier_frac=0.0005, outlier_mult=30.0,
                 weights=True)]
    return Workload(f"qwen72b-b{block}-{objective}", ts, block=block, objective=objective, fp8_div=256.0)


def workload(name: str) -> Workload:
    if name == "weight-2048":
        return Workload(name, [Tensor("w", 2048, 2048, "normal", 0, std=0.02)], block=16, objective="mse",
                        fp8_div=448.0)
    if name == "llama8b":
        return _llama8b()
    if name == "act-8192":
        return Workload(name, [Tensor("x", 8192, 4096, "student_t", 2000, outlier_count=16, outlier_mult=50.0)],
                        block=16, objective="mse", fp8_div=256.0, dynamic_scale=True)
    if name == "kvq":
        return _kvq()
    if name.startswith("qwen72b"):
        # qwen72b-b<block>-<objective>
        parts = name.split("-")
        block = int(parts[1][1:]) if len(parts) > 1 else 16
        objective = parts[2] if len(parts) > 2 else "mse"
        return _qwen72b(block, objective)
    if name.startswith("table7-"):
        b = int(name.split("-")[1])
        return Workload(name, [Tensor("x", b, 8192, "student_t", 5000 + b, outlier_count=16, outlier_mult=50.0)],
                        block=16, objective="mse", fp8_div=256.0, dynamic_scale=True)
    raise KeyError(name)


ALL_CONFIGS = ["weight-2048", "llama8b", "act-8192", "kvq"] + \
              [f"qwen72b-b{b}-{o}" for b in (16, 32, 64) for o in ("mse", "wmse")]


# ----------------------------------------------------------------------------- drawing
def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return g


def _outlier_cols(t: Tensor, g: torch.Generator) -> torch.Tensor:
    k = t.outlier_count if t.outlier_count is not None else int(round(t.outlier_frac * t.cols))
    if k <= 0:
        return torch.zeros(0, dtype=torch.long)
    return torch.randperm(t.cols, generator=g)[:k]


def draw(t: Tensor, rows: slice | None = None) -> torch.Tensor:
    """Draw the float32 values of tensor ``t`` (all rows, or a leading-row
    slice) and round them to bf16.  The full tensor is always drawn in the same
    order, so a row slice equals the same rows of the full draw."""
    g = _gen(t.seed)
    R, C = t.rows, t.cols
    if t.dist == "normal":
        x = torch.randn(R, C, generator=g, dtype=torch.float32) * t.std
    elif t.dist == "student_t":
        z = torch.randn(R, C, generator=g, dtype=torch.float32)
        chi = torch.zeros(R, C, dtype=torch.float32)
        for _ in range(3):
            n = torch.randn(R, C, generator=g, dtype=torch.float32)
            chi.add_(n * n)
        x = z / torch.sqrt(chi / 3.0)
    elif t.dist == "laplace":
        # u uniform on the open interval (-1/2, 1/2): rand() can return 0, which would give ln(0)
        u = torch.rand(R, C, generator=g, dtype=torch.float32).clamp_(min=2.0 ** -25).sub_(0.5)
        x = u.abs().mul_(-2.0).log1p_().mul_(-t.std)
        x.mul_(torch.sign(u))
        del u
    elif t.dist == "kvq":
        head_scale = torch.exp(0.5 * torch.randn(t.heads, generator=g, dtype=torch.float32))
        x = torch.randn(R, C, generator=g, dtype=torch.float32)
        # rows are [batch, head, seq] flattened with seq (4096) fastest
        seq = 4096 if R % (t.heads * 4096) == 0 else max(1, R // t.heads)
        idx = (torch.arange(R) // seq) % t.heads
        x.mul_(head_scale[idx].unsqueeze(1))
    else:
        raise KeyError(t.dist)
    cols = _outlier_cols(t, g)
    if cols.numel():
        x[:, cols] *= t.outlier_mult
    xb = x.to(torch.bfloat16)
    if rows is not None:
        xb = xb[rows].contiguous()
    return xb


def draw_weights(t: Tensor) -> torch.Tensor:
    """Per-input-channel WMSE weights, lognormal(0, 1), float32 [cols]
    (synthetic stand-in for the activation second moments ||X[:, i]||^2)."""
    g = _gen(t.seed + 500)
    return torch.exp(torch.randn(t.cols, generator=g, dtype=torch.float32))


def small_tensor(rows: int, cols: int, seed: int, dist: str = "normal", std: float = 0.02,
                 outliers: int = 0, mult: float = 20.0) -> torch.Tensor:
    """Small seeded bf16 tensor for parity tests (same distributions)."""
    t = Tensor("small", rows, cols, dist, seed, std=std, outlier_count=outliers, outlier_mult=mult,
               heads=1 if dist == "kvq" else 0)
    if dist == "kvq":
        g = _gen(seed)
        x = torch.randn(rows, cols, generator=g, dtype=torch.float32) * math.exp(0.5)
        return x.to(torch.bfloat16)
    return draw(t)
