"""The bench line's arithmetic (CPU): algorithmic bytes per weight of every
call (the roofline numerators), their totals over the 8B-shaped stack, the
fallback peaks, and the bookkeeping that ties recorded DRAM traffic to the
kernels' sources.  The per-weight figures are the ones the package format
fixes: a bf16 weight is 2 bytes, a 2-bit code a quarter byte per stage, and
each group of g weights carries one binary32 scale and zero per stage
(Eq. 2-3), or one binary16 scale on the symmetric grid."""
import os

import pytest

import bench
from paper_2608_04048_gb300 import workloads

N = 1 << 20


@pytest.mark.parametrize("g, per_weight", [(32, 4.0), (64, 3.5), (128, 3.25), (256, 3.125)])
def test_quantize_bytes_per_weight(g, per_weight):
    assert bench.alg_bytes_quantize(N, g) / N == per_weight


@pytest.mark.parametrize("k, per_weight", [(1, 2.3125), (2, 2.625), (3, 2.9375), (4, 3.25)])
def test_reconstruct_bytes_per_weight(k, per_weight):
    assert bench.alg_bytes_reconstruct(N, k, 128) / N == per_weight


def test_prefixes_and_step_bytes_per_weight():
    assert bench.alg_bytes_prefixes(N, 4, 128) / N == 9.25        # 4 planes + metadata, 4 bf16 outputs
    step = bench.alg_bytes_quantize(N, 128) + bench.STAGES * 2 * N  # package + every prefix
    assert step / N == 11.25
    assert bench.alg_bytes_quantize_sym16(N, 128) / N == 3.0625
    assert bench.alg_bytes_prefixes_sym16(N, 4, 128) / N == 9.0625


def test_stack_totals():
    specs = workloads.config_matrices("qwen3_8b_stack")
    q = sum(bench.alg_bytes_quantize(sp.numel, sp.group) for sp in specs)
    assert round(q / 1e9, 2) == 22.57
    rec = [round(sum(bench.alg_bytes_reconstruct(sp.numel, k, sp.group) for sp in specs) / 1e9, 2)
           for k in (1, 2, 3, 4)]
    assert rec == [16.06, 18.23, 20.40, 22.57]
    assert sum(2 * sp.numel for sp in specs) == 13_891_534_848  # the stack's bf16 bytes


def test_fallback_peaks(monkeypatch, tmp_path):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))  # no MEASURED_PEAKS.json there
    p = bench.measured_peaks()
    assert (p["hbm_gbs"], p["bf16_tflops"], p["source"]) == (6800.0, 1900.0, "fallback")


def test_traffic_bookkeeping_names_existing_sources():
    csrc = os.path.join(bench.ROOT, "paper_2608_04048_gb300", "csrc")
    assert set(bench.TRAFFIC_KERNELS) <= set(bench.KERNEL_SOURCES)
    for name, files in bench.KERNEL_SOURCES.items():
        for f in files:
            assert os.path.exists(os.path.join(csrc, f)), (name, f)
        assert len(bench.kernel_source_hash(name)) == 64
    # per-weight bytes behind each recorded entry agree with the formulas
    assert bench.TRAFFIC_KERNELS["rrq_quantize"][1] == 3.25
    assert bench.TRAFFIC_KERNELS["rrq_reconstruct_prefixes"][1] == 9.25
    assert bench.TRAFFIC_KERNELS["rrq_reconstruct_k4"][1] == 3.25
    assert bench.TRAFFIC_KERNELS["rrq_quantize_prefixes"][1] == 11.25


def test_rank_seed_offsets_leave_the_stack_seed_range():
    seeds = {sp.seed for sp in workloads.config_matrices("qwen3_8b_stack")}
    for r in range(1, 8):
        assert not seeds & {s + bench.shard_seed_offset(r) for s in seeds}
