"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times (rrq_quantize_batch / rrq_reconstruct_batch over whole
stacks): the oracle recomputes sampled groups of every matrix (groups are
independent, so a sampled group's codes, scale, zero and reconstruction are
exactly those of the full run), plus whole small matrices.

Workloads (see paper_2608_04048_gb300.workloads): a 4096x4096 matrix, one
Qwen3-8B-shaped layer, the full 36-layer Qwen3-8B-shaped stack, the
8192x8192 distribution x group-size sweep, and full-size Qwen3-32B-shaped
layers."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bf16_bits, check_full, check_sampled, sample_groups

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)


def _batched(specs, group=128, stages=4, seed_offset=0):
    mats = [workloads.generate_spec(sp, "cuda") if seed_offset == 0 else
            workloads.generate(sp.rows, sp.cols, sp.seed + seed_offset, sp.dist, "cuda") for sp in specs]
    pkgs = binding.rrq_quantize_batch(mats, group=group, n_stages=stages)
    return mats, pkgs


def test_qwen3_8b_layer_full_and_sampled():
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats, pkgs = _batched(specs)
    torch.cuda.synchronize()
    for i, (sp, W, pkg) in enumerate(zip(specs, mats, pkgs)):
        if sp.numel <= 1024 * 4096:  # k_proj, v_proj: whole matrices
            ref = oracle.quantize(bf16_bits(W), 128, 4)
            from gpu_helpers import assert_package_equal, gpu_package_host
            assert_package_equal(gpu_package_host(pkg), ref, 4, sp.name)
        idx = sample_groups(sp.numel // 128, 4000, seed=i)
        check_sampled(W, pkg, idx, where=sp.name)


def test_qwen3_8b_stack_bench_configuration():
    """The benchmark's workload exactly: 252 matrices (6.95e9 weights) in
    batched launches; 384 sampled groups of every matrix checked against
    the oracle at every prefix."""
    specs = workloads.config_matrices("qwen3_8b_stack")
    mats, pkgs = _batched(specs)
    outs = {k: binding.rrq_reconstruct_batch(pkgs, k) for k in (1, 2, 3, 4)}
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    for i, (sp, W, pkg) in enumerate(zip(specs, mats, pkgs)):
        idx = sample_groups(sp.numel // 128, 256, seed=1000 + i)
        it = torch.from_numpy(idx).cuda()
        Wg = W.reshape(-1, 128).index_select(0, it)
        ref = oracle.quantize(bf16_bits(Wg), 128, 4)
        for k in range(4):
            gc = pkg.codes[k].view(-1, 32).index_select(0, it).cpu().numpy().reshape(-1)
            assert np.array_equal(gc, ref[0][k]), f"{sp.name} stage {k} codes"
            gs = pkg.scales[k].index_select(0, it).cpu().numpy()
            gz = pkg.zeros[k].index_select(0, it).cpu().numpy()
            assert np.array_equal(gs.view(np.uint32), ref[1][k].view(np.uint32)), f"{sp.name} stage {k} scales"
            assert np.array_equal(gz.view(np.uint32), ref[2][k].view(np.uint32)), f"{sp.name} stage {k} zeros"
        for k in (1, 2, 3, 4):
            got = bf16_bits(outs[k][i].reshape(-1, 128).index_select(0, it))
            want = oracle.reconstruct(*ref, idx.size, 128, 128, k)
            assert np.array_equal(got, want), f"{sp.name} reconstruct k={k}"
    del mats, pkgs, outs
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dist", ["normal", "t3", "t3_col0.001", "t3_col0.01"])
def test_sweep_8192_all_groups(dist):
    """8192x8192, one input per distribution, group sizes 32/64/128/256."""
    specs = [sp for sp in workloads.config_matrices("sweep_8192") if sp.dist == dist]
    W = workloads.generate_spec(specs[0], "cuda")
    for sp in specs:
        pkg = binding.rrq_quantize(W, sp.group, 4)
        idx = sample_groups(sp.numel // sp.group, 3000, seed=sp.group)
        check_sampled(W, pkg, idx, where=f"{dist} g{sp.group}")
        del pkg


def test_qwen3_32b_layers():
    """Full-size Qwen3-32B-shaped layers 0 and 63 (14 matrices, the largest
    25600x5120), batched; sampled groups against the oracle."""
    specs = [sp for sp in workloads.config_matrices("qwen3_32b_stack")
             if sp.name.startswith(("layers.0.", "layers.63."))]
    mats, pkgs = _batched(specs)
    torch.cuda.synchronize()
    for i, (sp, W, pkg) in enumerate(zip(specs, mats, pkgs)):
        idx = sample_groups(sp.numel // 128, 2000, seed=5000 + i)
        check_sampled(W, pkg, idx, where=sp.name)


def test_single_4096_is_seed_0_normal():
    sp = workloads.config_matrices("single_4096")[0]
    assert (sp.rows, sp.cols, sp.seed, sp.dist) == (4096, 4096, 0, "normal")
    W = workloads.generate_spec(sp, "cuda")
    check_full(W, 128, 4, where="single_4096")
