"""GPU parity of the one-prefix reconstruction of matrices made of whole
2048-weight chunks (the wide-lane kernel; Eq. 8, Appendix C): every package
format and group size, every prefix k = 1..4, in batches whose chunks belong
to several matrices.  The kernel brings the package in by bulk copies up to
k = 2 and by per-lane 16-byte copies from k = 3, with a slot layout that
depends on the format and group (scale and zero arrays of 2048/g entries),
so each combination is its own case.  Outputs are compared with the oracle
bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import _cmp_bytes, assert_package_equal, bf16_bits, gpu_package_host, scales_host

pytestmark = pytest.mark.gpu

GROUPS = (32, 64, 128, 256)
# every size a multiple of 2048 weights: 2048, 96 and 1 chunk(s) of 2048 x 2
SHAPES = [(1024, 4096), (96, 2048), (8, 256)]
FORMATS = {
    "asym_f32": (binding.GRID_ASYM, binding.SCALE_F32),
    "sym_f32": (binding.GRID_SYM, binding.SCALE_F32),
    "sym_f16": (binding.GRID_SYM, binding.SCALE_F16),
}


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)
    yield


@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("fmt", sorted(FORMATS))
def test_whole_chunk_batches_every_prefix(fmt, group):
    grid, scale_type = FORMATS[fmt]
    mats = [workloads.generate(r, c, 41 * i + group, "t3_rowout", "cuda") for i, (r, c) in enumerate(SHAPES)]
    assert all(W.numel() % 2048 == 0 for W in mats)
    pkgs = binding.rrq_quantize_ex(mats, group, 4, grid, scale_type)
    refs = []
    for i, (W, pkg) in enumerate(zip(mats, pkgs)):
        if fmt == "asym_f32":
            ref = oracle.quantize(bf16_bits(W), group, 4)
            assert_package_equal(gpu_package_host(pkg), ref, 4, f"{fmt} g{group} item {i}")
        else:
            f16 = fmt == "sym_f16"
            ref = oracle.quantize_sym(bf16_bits(W), group, 4, f16)
            gs = scales_host(pkg)
            for s in range(4):
                _cmp_bytes(pkg.codes[s].cpu().numpy(), ref[0][s], f"{fmt} g{group} item {i} stage {s} codes")
                _cmp_bytes(gs[s], ref[1][s], f"{fmt} g{group} item {i} stage {s} scales")
        refs.append(ref)
    for k in (1, 2, 3, 4):
        outs = binding.rrq_reconstruct_ex(pkgs, k)
        torch.cuda.synchronize()
        assert binding.rrq_get_device_status() == 0
        for i, (W, ref) in enumerate(zip(mats, refs)):
            rows, cols = W.shape
            if fmt == "asym_f32":
                want = oracle.reconstruct(*ref, rows, cols, group, k)
            else:
                want = oracle.reconstruct_sym(ref[0], ref[1], rows, cols, group, k, fmt == "sym_f16")
            got = bf16_bits(outs[i][0])
            if not np.array_equal(got, want):
                bad = np.nonzero(got.reshape(-1) != want.reshape(-1))[0]
                raise AssertionError(f"{fmt} g{group} item {i} k={k}: {bad.size} mismatches, first at {bad[0]}")
