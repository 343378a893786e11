"""GPU parity for the build with prefixes (rrq_quantize_prefixes: Algorithm 1
and Eq. 8 at every prefix in one pass): for every format and group size the
package and every bf16 prefix equal the CPU oracle's on ragged shapes, bit for
bit; and they equal rrq_quantize_ex's package and rrq_reconstruct_ex's
prefixes on it (the two-call path).  The whole-workload checks of the same
call are in test_gpu_full_size.py."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bf16_bits, scales_host
from test_gpu_parity import _edge_matrix

pytestmark = pytest.mark.gpu

GROUPS = (32, 64, 128, 256)
FORMATS = [(binding.GRID_ASYM, binding.SCALE_F32), (binding.GRID_SYM, binding.SCALE_F32),
           (binding.GRID_SYM, binding.SCALE_F16)]
FMT_IDS = ["asym_f32", "sym_f32", "sym_f16"]


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)
    yield
    binding.rrq_set_debug_flags(0)


def _same(a, b):
    return torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8))


def check(mats, group, S, fmt, where=""):
    pkgs, outs = binding.rrq_quantize_prefixes(mats, group, S, *fmt)
    refs = binding.rrq_quantize_ex(mats, group, S, *fmt)
    routs = binding.rrq_reconstruct_ex(refs, S, all_prefixes=True)
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
    for i, (p, r) in enumerate(zip(pkgs, refs)):
        for k in range(S):
            assert _same(p.codes[k], r.codes[k]), f"{where} item {i} stage {k} codes"
            assert _same(p.scales[k], r.scales[k]), f"{where} item {i} stage {k} scales"
            if p.zeros:
                assert _same(p.zeros[k], r.zeros[k]), f"{where} item {i} stage {k} zeros"
            assert _same(outs[i][k], routs[i][k]), f"{where} item {i} prefix {k + 1}"
    return pkgs, outs


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", GROUPS)
def test_formats_and_groups(group, fmt):
    mats = [workloads.generate(133, 5 * group, 31 + group, d, "cuda") for d in ("t3_rowout", "normal")]
    check(mats, group, 4, fmt, where=f"g{group} {fmt}")


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
def test_fewer_stages_and_shapes(fmt):
    for shape in ((1, 32), (31, 32), (7, 2304), (2049, 128)):
        for g in GROUPS:
            if shape[1] % g:
                continue
            for S in (1, 2, 3):
                W = workloads.generate(shape[0], shape[1], S + shape[0], "t3", "cuda")
                check([W], g, S, fmt, where=f"{shape} g{g} S{S}")


@pytest.mark.parametrize("group", GROUPS)
def test_edge_groups_and_forced_exact(group):
    W = _edge_matrix(24, 8 * group, group, seed=300 + group)
    check([W], group, 4, FORMATS[0], where=f"edge g{group}")
    binding.rrq_set_debug_flags(1)
    try:
        for fmt in FORMATS:
            Wf = W if fmt[1] == binding.SCALE_F32 else workloads.generate(24, 8 * group, 3, "t3_rowout", "cuda")
            check([Wf], group, 4, fmt, where=f"forced exact g{group} {fmt}")
    finally:
        binding.rrq_set_debug_flags(0)


def _oracle_package(W, group, S, fmt):
    """(codes, scales as stored, zeros or None) and the prefixes 1..S."""
    bits = bf16_bits(W)
    rows, cols = W.shape
    if fmt[0] == binding.GRID_ASYM:
        codes, scales, zeros = oracle.quantize(bits, group, S)
        pre = [oracle.reconstruct(codes, scales, zeros, rows, cols, group, k) for k in range(1, S + 1)]
    else:
        f16 = fmt[1] == binding.SCALE_F16
        codes, scales = oracle.quantize_sym(bits, group, S, f16)
        zeros = None
        pre = [oracle.reconstruct_sym(codes, scales, rows, cols, group, k, f16) for k in range(1, S + 1)]
    return codes, scales, zeros, pre


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", GROUPS)
def test_each_format_against_the_oracle(group, fmt):
    """Every output of rrq_quantize_prefixes against the oracle directly:
    ragged shapes (a single group, chunk tails that end mid-warp, a matrix of
    many chunks), heavy tails and outliers, 4 and 3 stages."""
    shapes = [(1, group), (7, 3 * group), (33, 5 * group), (130, 2 * group), (5, 4096 // group * group)]
    for S in (4, 3):
        mats = [workloads.generate(r, c, 70 + 3 * i + S, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
        pkgs, outs = binding.rrq_quantize_prefixes(mats, group, S, *fmt)
        torch.cuda.synchronize()
        assert binding.rrq_get_device_status() == 0
        for i, (W, p) in enumerate(zip(mats, pkgs)):
            codes, scales, zeros, pre = _oracle_package(W, group, S, fmt)
            where = f"g{group} S{S} {shapes[i]}"
            for k in range(S):
                assert np.array_equal(p.codes[k].cpu().numpy(), codes[k]), f"{where} stage {k} codes"
                got = p.scales[k].cpu().numpy()
                assert np.array_equal(got.view(np.uint8), np.ascontiguousarray(scales[k]).view(np.uint8)), \
                    f"{where} stage {k} scales"
                if zeros is not None:
                    assert np.array_equal(p.zeros[k].cpu().numpy().view(np.uint32), zeros[k].view(np.uint32)), \
                        f"{where} stage {k} zeros"
                assert np.array_equal(bf16_bits(outs[i][k]), pre[k]), f"{where} prefix {k + 1}"


def test_against_oracle_and_across_launches():
    rng = np.random.default_rng(31)
    shapes = [(int(rng.integers(1, 30)), 128 * int(rng.integers(1, 10))) for _ in range(70)]
    mats = [workloads.generate(r, c, 2000 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs, outs = check(mats, 128, 4, FORMATS[0], where="batch")
    for i in (0, 33, 69):
        W = mats[i]
        ref = oracle.quantize(bf16_bits(W), 128, 4)
        for k in range(1, 5):
            want = oracle.reconstruct(*ref, W.shape[0], W.shape[1], 128, k)
            assert np.array_equal(bf16_bits(outs[i][k - 1]), want), f"item {i} prefix {k}"


def test_errors():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize_prefixes([W], 128, 2, outs=[[torch.empty(0, dtype=torch.bfloat16, device="cuda")] * 2])
    assert e.value.status == 1
    pkg = binding.Package.empty(8, 256, 128, 2)
    o = torch.empty((8, 256), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.RRQError) as e:  # two prefixes into one buffer
        binding.rrq_quantize_prefixes([W], 128, 2, pkgs=[pkg], outs=[[o, o]])
    assert e.value.status == 1
