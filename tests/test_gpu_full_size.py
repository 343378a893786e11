"""GPU parity at the workloads' full sizes: EVERY output compared with the
CPU oracle, which runs over all host cores (tests/full_parity.py,
oracle/pool.py).  Algorithm 1 and Eq. 8: packed codes, scales and zeros bit
for bit, bf16 prefixes with 0 ULP.

Workloads (paper_2608_04048_gb300.workloads):
- a 4096x4096 normal matrix (seed 0);
- one Qwen3-8B-shaped layer, in all three package formats, through
  rrq_quantize_prefixes (the package and every prefix in one pass);
- the whole 36-layer Qwen3-8B-shaped stack (252 matrices, 6.95e9 weights)
  through exactly the call bench.py times: one rrq_quantize_prefixes over
  all 252 matrices (launches of 64, 64, 64 and 60 matrices);
- the 8192x8192 sweep: four distributions x groups 32/64/128/256;
- the whole 64-layer Qwen3-32B-shaped stack (448 matrices, 3.12e10 weights)
  through rrq_quantize_batch, and rrq_reconstruct_batch at k = 1..4 of each
  layer into reused buffers (the four prefixes of the whole stack do not
  fit in HBM beside it)."""
import pytest
import torch

from oracle.pool import OraclePool
from paper_2608_04048_gb300 import binding, build, workloads
from full_parity import Entry, Unit, check_units
from gpu_helpers import check_full

pytestmark = pytest.mark.gpu

FORMATS = {"asym_f32": (binding.GRID_ASYM, binding.SCALE_F32), "sym_f32": (binding.GRID_SYM, binding.SCALE_F32),
           "sym_f16": (binding.GRID_SYM, binding.SCALE_F16)}


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)


@pytest.fixture(scope="module")
def pool():
    with OraclePool() as p:
        yield p


def _prefix_units(specs, mats, pkgs, outs, per: int):
    return [Unit([Entry(specs[j].name, mats[j], pkgs[j], outs[j]) for j in range(i, min(i + per, len(specs)))])
            for i in range(0, len(specs), per)]


def _assert_equal(summary):
    assert not summary["mismatches"], "\n".join(summary["mismatches"])


def test_single_4096_is_seed_0_normal():
    sp = workloads.config_matrices("single_4096")[0]
    assert (sp.rows, sp.cols, sp.seed, sp.dist) == (4096, 4096, 0, "normal")
    W = workloads.generate_spec(sp, "cuda")
    check_full(W, 128, 4, where="single_4096")


@pytest.mark.parametrize("fmt", list(FORMATS))
def test_qwen3_8b_layer_every_output(fmt, pool):
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs, outs = binding.rrq_quantize_prefixes(mats, 128, 4, *FORMATS[fmt])
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    _assert_equal(check_units(f"qwen3_8b_layer {fmt} (rrq_quantize_prefixes)",
                              _prefix_units(specs, mats, pkgs, outs, 7), pool))


def test_qwen3_8b_stack_every_output_of_the_timed_call(pool):
    """The benchmark's step exactly: the 252 matrices in one
    rrq_quantize_prefixes call, every code, scale, zero and prefix checked."""
    specs = workloads.config_matrices("qwen3_8b_stack")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = [binding.Package.empty(sp.rows, sp.cols, 128, 4) for sp in specs]
    outs = [[torch.empty((sp.rows, sp.cols), dtype=torch.bfloat16, device="cuda") for _ in range(4)]
            for sp in specs]
    items = binding.quantize_prefixes_descs(mats, pkgs, outs)
    binding.rrq_quantize_prefixes(mats, 128, 4, binding.GRID_ASYM, binding.SCALE_F32, pkgs, outs,
                                  torch.cuda.current_stream(), items)
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    summary = check_units("qwen3_8b_stack (the timed rrq_quantize_prefixes call)",
                          _prefix_units(specs, mats, pkgs, outs, 7), pool)
    assert summary["weights"] == sum(sp.numel for sp in specs)
    del mats, pkgs, outs, items
    torch.cuda.empty_cache()
    _assert_equal(summary)


def test_sweep_8192_every_output(pool):
    """8192x8192, one input per distribution, groups 32/64/128/256, through
    rrq_quantize_prefixes (package and every prefix)."""
    specs = workloads.config_matrices("sweep_8192")
    units = []
    keep = []
    inputs = {}
    for sp in specs:
        if sp.dist not in inputs:
            inputs[sp.dist] = workloads.generate_spec(sp, "cuda")
        W = inputs[sp.dist]
        pkgs, outs = binding.rrq_quantize_prefixes([W], sp.group, 4)
        keep.append((pkgs, outs))
        units.append(Unit([Entry(sp.name, W, pkgs[0], outs[0])]))
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    _assert_equal(check_units("sweep_8192 (4 distributions x 4 groups, rrq_quantize_prefixes)", units, pool))


def test_qwen3_32b_stack_every_output(pool):
    """All 64 Qwen3-32B-shaped layers: rrq_quantize_batch over the 448
    matrices (launches of 64), then per layer rrq_reconstruct_batch at each
    k into one reused buffer per matrix; every output checked."""
    specs = workloads.config_matrices("qwen3_32b_stack")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    bufs = [torch.empty((sp.rows, sp.cols), dtype=torch.bfloat16, device="cuda") for sp in specs[:7]]
    units = []
    for i in range(0, len(specs), 7):
        layer = list(range(i, i + 7))
        def recon(k, layer=layer):
            return binding.rrq_reconstruct_batch([pkgs[j] for j in layer], k, outs=bufs)
        units.append(Unit([Entry(specs[j].name, mats[j], pkgs[j]) for j in layer], (1, 2, 3, 4), recon))
    summary = check_units("qwen3_32b_stack (rrq_quantize_batch + rrq_reconstruct_batch k=1..4)", units, pool)
    assert binding.rrq_get_device_status() == 0
    assert summary["weights"] == sum(sp.numel for sp in specs)
    del mats, pkgs, bufs, units
    torch.cuda.empty_cache()
    _assert_equal(summary)
