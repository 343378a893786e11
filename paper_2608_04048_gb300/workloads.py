"""Seeded synthetic weight matrices shaped like the paper's models.

This module generates inputs only: it holds none of the quantization
arithmetic, and both the CUDA path and the CPU oracle receive the same tensors
from it.  The paper's checkpoints (Qwen3-8B, Qwen3-32B, Section 5.1) are not
available, so seeded stand-ins take their linear-layer shapes and a weight
distribution with the heavy tails and rare large outliers the paper measures
(Section 3 peak-to-mean ratio; Appendix F, Table 9).

Distributions (sigma = 0.02):
  normal      i.i.d. N(0, sigma^2)
  t3          Student-t with 3 degrees of freedom scaled to std sigma, built
              from normals: z0 / sqrt((z1^2 + z2^2 + z3^2) / 3) * sigma / sqrt(3)
  t3_rowout   t3 plus, in every row, round(0.001 * cols) distinct random
              columns set to +-20 sigma = +-0.4 with random sign
  t3_col{p}   t3 plus a fixed seeded set of round(p * cols) columns whose
              entries in every row are set to +-0.4 with random sign
Values are drawn in fp32 on the requested device and rounded to bf16
(round-to-nearest-even), like bf16 checkpoints.
"""
from __future__ import annotations

import hashlib
import math
from dataclasses import dataclass

import torch

SIGMA = 0.02
OUTLIER = 20 * SIGMA

# (name, out_features, in_features) of one decoder layer's linear layers
QWEN3_8B_LAYER = [
    ("q_proj", 4096, 4096), ("k_proj", 1024, 4096), ("v_proj", 1024, 4096),
    ("o_proj", 4096, 4096), ("gate_proj", 12288, 4096), ("up_proj", 12288, 4096),
    ("down_proj", 4096, 12288),
]
QWEN3_32B_LAYER = [
    ("q_proj", 8192, 5120), ("k_proj", 1024, 5120), ("v_proj", 1024, 5120),
    ("o_proj", 5120, 8192), ("gate_proj", 25600, 5120), ("up_proj", 25600, 5120),
    ("down_proj", 5120, 25600),
]


@dataclass(frozen=True)
class MatrixSpec:
    name: str
    rows: int
    cols: int
    seed: int
    dist: str
    group: int = 128

    @property
    def numel(self) -> int:
        return self.rows * self.cols


def config_matrices(config: str) -> list[MatrixSpec]:
    """The matrices of one named workload.

    single_4096      one 4096x4096 normal matrix, seed 0
    qwen3_8b_layer   one Qwen3-8B-shaped layer, t3_rowout, seeds 2000+m
    qwen3_8b_stack   36 such layers, seeds 3000 + 7*layer + m
    sweep_8192       8192x8192 x {normal, t3, t3_col0.001, t3_col0.01} x
                     group {32, 64, 128, 256}, seeds 4000 + distribution index
    qwen3_32b_stack  64 Qwen3-32B-shaped layers, seeds 5000 + 7*layer + m
    """
    if config == "single_4096":
        return [MatrixSpec("w", 4096, 4096, 0, "normal")]
    if config == "qwen3_8b_layer":
        return [MatrixSpec(n, r, c, 2000 + m, "t3_rowout") for m, (n, r, c) in enumerate(QWEN3_8B_LAYER)]
    if config == "qwen3_8b_stack":
        return [MatrixSpec(f"layers.{l}.{n}", r, c, 3000 + 7 * l + m, "t3_rowout")
                for l in range(36) for m, (n, r, c) in enumerate(QWEN3_8B_LAYER)]
    if config == "sweep_8192":
        dists = ["normal", "t3", "t3_col0.001", "t3_col0.01"]
        return [MatrixSpec(f"{d}.g{g}", 8192, 8192, 4000 + i, d, g)
                for i, d in enumerate(dists) for g in (32, 64, 128, 256)]
    if config == "qwen3_32b_stack":
        return [MatrixSpec(f"layers.{l}.{n}", r, c, 5000 + 7 * l + m, "t3_rowout")
                for l in range(64) for m, (n, r, c) in enumerate(QWEN3_32B_LAYER)]
    raise ValueError(f"unknown workload {config!r}")


def _t3(shape, gen, device):
    z = torch.randn((4,) + tuple(shape), generator=gen, device=device, dtype=torch.float32)
    t = z[0] / torch.sqrt((z[1] * z[1] + z[2] * z[2] + z[3] * z[3]) / 3.0)
    return t * (SIGMA / math.sqrt(3.0))


def generate(rows: int, cols: int, seed: int, dist: str = "normal",
             device="cpu") -> torch.Tensor:
    """A bf16 [rows, cols] matrix drawn from `dist` with generator seed `seed`."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    if dist == "normal":
        w = torch.randn((rows, cols), generator=gen, device=device, dtype=torch.float32) * SIGMA
    elif dist == "t3" or dist == "t3_rowout" or dist.startswith("t3_col"):
        w = _t3((rows, cols), gen, device)
    else:
        raise ValueError(f"unknown distribution {dist!r}")
    if dist == "t3_rowout":
        m = round(0.001 * cols)
        if m > 0:
            keys = torch.rand((rows, cols), generator=gen, device=device)
            idx = keys.topk(m, dim=1).indices
            del keys
            sign = torch.randint(0, 2, (rows, m), generator=gen, device=device).to(torch.float32) * 2 - 1
            w.scatter_(1, idx, sign * OUTLIER)
    elif dist.startswith("t3_col"):
        p = float(dist[len("t3_col"):])
        m = round(p * cols)
        if m > 0:
            colidx = torch.randperm(cols, generator=gen, device=device)[:m]
            sign = torch.randint(0, 2, (rows, m), generator=gen, device=device).to(torch.float32) * 2 - 1
            w[:, colidx] = sign * OUTLIER
    return w.to(torch.bfloat16)


def generate_spec(spec: MatrixSpec, device="cpu") -> torch.Tensor:
    return generate(spec.rows, spec.cols, spec.seed, spec.dist, device)


def sha256_bf16(w: torch.Tensor) -> str:
    """SHA-256 of a bf16 tensor's bytes (row-major), for input manifests."""
    b = w.detach().contiguous().view(torch.int16).cpu().numpy().tobytes()
    return hashlib.sha256(b).hexdigest()


def pmr_report(w: torch.Tensor, group: int = 128) -> dict:
    """Input-realism statistic (Section 3): peak-to-mean ratio max|w| /
    mean|w| per group; the tensor-wise maximum over groups and the mean of
    the groupwise values.  Reported beside the paper's real-model figures,
    not used by the quantizer."""
    a = w.float().abs().reshape(-1, group)
    pmr = a.max(dim=1).values / a.mean(dim=1).clamp_min(1e-30)
    return {"max_group_pmr": float(pmr.max()), "mean_group_pmr": float(pmr.mean())}
