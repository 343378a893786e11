"""The seeded synthetic inputs (CPU): the workloads' shapes, sizes and seed
schemes, determinism by seed, and the recipe of each distribution (outlier
counts and values, spread), so that the inputs both the CUDA path and the
oracle receive are the ones the measurement claims.  Shapes follow the
Qwen3-8B and Qwen3-32B linear layers of Section 5.1; the peak-to-mean
statistic is the one of Section 3."""
import math

import numpy as np
import pytest
import torch

from paper_2608_04048_gb300 import workloads

OUT = float(torch.tensor(workloads.OUTLIER).to(torch.bfloat16))  # +-0.4 as bf16


@pytest.mark.parametrize("config, count, weights", [
    ("single_4096", 1, 16_777_216),
    ("qwen3_8b_layer", 7, 192_937_984),
    ("qwen3_8b_stack", 252, 6_945_767_424),
    ("sweep_8192", 16, 16 * 67_108_864),
    ("qwen3_32b_stack", 448, 31_205_621_760),
])
def test_config_sizes(config, count, weights):
    specs = workloads.config_matrices(config)
    assert len(specs) == count
    assert sum(sp.numel for sp in specs) == weights


def test_config_seeds_and_groups():
    layer = workloads.config_matrices("qwen3_8b_layer")
    assert [sp.seed for sp in layer] == list(range(2000, 2007))
    stack = workloads.config_matrices("qwen3_8b_stack")
    assert [sp.seed for sp in stack] == [3000 + 7 * l + m for l in range(36) for m in range(7)]
    assert len({sp.seed for sp in stack}) == 252
    big = workloads.config_matrices("qwen3_32b_stack")
    assert [sp.seed for sp in big] == [5000 + 7 * l + m for l in range(64) for m in range(7)]
    sweep = workloads.config_matrices("sweep_8192")
    assert {(sp.dist, sp.group, sp.seed) for sp in sweep} == {
        (d, g, 4000 + i) for i, d in enumerate(["normal", "t3", "t3_col0.001", "t3_col0.01"])
        for g in (32, 64, 128, 256)}
    assert all(sp.group == 128 for sp in stack + big + layer)
    with pytest.raises(ValueError):
        workloads.config_matrices("no_such_workload")


@pytest.mark.parametrize("dist", ["normal", "t3", "t3_rowout", "t3_col0.01"])
def test_deterministic_by_seed(dist):
    a = workloads.generate(16, 1024, 7, dist)
    b = workloads.generate(16, 1024, 7, dist)
    c = workloads.generate(16, 1024, 8, dist)
    assert a.dtype == torch.bfloat16 and a.shape == (16, 1024)
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    assert workloads.sha256_bf16(a) == workloads.sha256_bf16(b) != workloads.sha256_bf16(c)


def test_row_outliers_exact_count_and_value():
    rows, cols = 64, 4096
    w = workloads.generate(rows, cols, 11, "t3_rowout").float()
    m = round(0.001 * cols)
    is_out = w.abs() == OUT
    assert (is_out.sum(dim=1) == m).all()
    assert set(w[is_out].unique().tolist()) <= {OUT, -OUT}
    # both signs occur, and the columns differ between rows
    assert (w[is_out] > 0).any() and (w[is_out] < 0).any()
    assert len({tuple(np.nonzero(r)[0]) for r in is_out.numpy()}) > rows // 2


@pytest.mark.parametrize("p", [0.001, 0.01])
def test_column_outliers_shared_by_every_row(p):
    rows, cols = 32, 8192
    w = workloads.generate(rows, cols, 12, f"t3_col{p}").float()
    full_cols = (w.abs() == OUT).all(dim=0)
    assert int(full_cols.sum()) == round(p * cols)
    # the rest of the matrix is plain t3 (no value of exactly +-0.4 elsewhere)
    assert int((w[:, ~full_cols].abs() == OUT).sum()) == 0


def test_spread_of_normal_and_t3():
    n = 1 << 20
    z = workloads.generate(1024, 1024, 3, "normal").float().reshape(-1)
    assert abs(float(z.std()) / workloads.SIGMA - 1) < 0.01
    assert abs(float(z.mean())) < 0.001
    t = workloads.generate(1024, 1024, 4, "t3").float().reshape(-1)
    # Student-t(3) scaled to std sigma: scale sigma / sqrt(3); its quartiles
    # are +-0.764892 scale (the t3 quantile at 0.75)
    q1, q3 = np.quantile(t.numpy(), [0.25, 0.75])
    want = 0.764892 * workloads.SIGMA / math.sqrt(3.0)
    assert abs(q3 / want - 1) < 0.02 and abs(-q1 / want - 1) < 0.02
    assert t.numel() == n


def test_pmr_closed_forms():
    g = 128
    one = torch.zeros((2, g))
    one[0, 5] = 0.5                      # one nonzero: max / mean = g
    one[1, :] = 0.25                     # constant: 1
    r = workloads.pmr_report(one.to(torch.bfloat16), g)
    assert r["max_group_pmr"] == pytest.approx(g)
    assert r["mean_group_pmr"] == pytest.approx((g + 1) / 2)
