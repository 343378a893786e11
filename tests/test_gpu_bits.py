"""GPU parity for heterogeneous stage widths (Section 3.2's per-stage
formats; the 1+3 / 2+2 / 3+1 splits of Table 3) through rrq_quantize_ex /
rrq_reconstruct_ex on the asymmetric grid: codes (packed LSB-first at b_k
bits), scales and zeros bit for bit, every prefix with 0 ULP; and the group
peak-to-mean ratio (rrq_group_pmr, the K/MAE statistic of Table 9) within the
bound of its binary32 sum."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bf16_bits

pytestmark = pytest.mark.gpu

GROUPS = (32, 64, 128, 256)
SPLITS = [(1, 3), (3, 1), (1, 1, 1, 1), (4, 4), (4, 2, 1, 3), (2, 2), (3, 3, 2)]


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)
    yield
    binding.rrq_set_debug_flags(0)


def check_bits(W, group, bits, where=""):
    rows, cols = W.shape
    S = len(bits)
    (pkg,) = binding.rrq_quantize_ex([W], group, S, binding.GRID_ASYM, binding.SCALE_F32, bits=list(bits))
    torch.cuda.synchronize()
    rc, rs, rz = oracle.quantize_bits(bf16_bits(W), group, list(bits))
    for k in range(S):
        got = pkg.codes[k].cpu().numpy()
        assert got.nbytes == rc[k].nbytes, f"{where} stage {k} code bytes"
        if not np.array_equal(got, rc[k]):
            bad = np.nonzero(got != rc[k])[0]
            raise AssertionError(f"{where} stage {k} codes: {bad.size} bytes differ, first {bad[0]}")
        assert np.array_equal(pkg.scales[k].cpu().numpy().view(np.uint32), rs[k].view(np.uint32)), f"{where} stage {k} scales"
        assert np.array_equal(pkg.zeros[k].cpu().numpy().view(np.uint32), rz[k].view(np.uint32)), f"{where} stage {k} zeros"
    allp = binding.rrq_reconstruct_ex([pkg], S, all_prefixes=True)[0]
    for k in range(1, S + 1):
        one = binding.rrq_reconstruct_ex([pkg], k)[0][0]
        torch.cuda.synchronize()
        want = oracle.reconstruct_bits(rc, rs, rz, rows, cols, group, k, list(bits))
        assert np.array_equal(bf16_bits(one), want), f"{where} prefix {k}"
        assert np.array_equal(bf16_bits(allp[k - 1]), want), f"{where} all-prefix {k}"
    return pkg


@pytest.mark.parametrize("bits", SPLITS, ids=lambda b: "+".join(map(str, b)))
@pytest.mark.parametrize("group", GROUPS)
def test_splits_and_groups(group, bits):
    W = workloads.generate(133, 5 * group, 90 + group, "t3_rowout", "cuda")
    check_bits(W, group, bits, where=f"g{group} {bits}")


@pytest.mark.parametrize("shape", [(1, 32), (3, 96), (31, 32), (7, 2304), (2049, 128)])
def test_shapes(shape):
    rows, cols = shape
    for g in GROUPS:
        if cols % g:
            continue
        for bits in ((1, 3), (4, 2, 1, 3)):
            W = workloads.generate(rows, cols, rows + cols + len(bits), "t3", "cuda")
            check_bits(W, g, bits, where=f"{shape} g{g} {bits}")


def _tie_matrix(rows, cols, group, b, seed):
    """Groups on a 2^b-level grid including half steps (exact ties for the
    rounding), plus Gaussian groups: exercises the per-element fallback."""
    rng = np.random.default_rng(seed)
    steps = (1 << b) - 1
    out = []
    for gi in range(rows * cols // group):
        if gi % 2:
            x = rng.normal(0, 0.02, group)
        else:
            a, d = int(rng.integers(-40, 40)), int(rng.integers(1, 16))
            q = rng.integers(0, 2 * steps + 1, group) / 2.0
            q[0], q[-1] = 0, steps
            x = (a + q * d) / 1024.0
        out.append(x.astype(np.float32))
    u = np.concatenate(out).view(np.uint32)
    bits16 = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    return torch.from_numpy(bits16.reshape(rows, cols).view(np.int16)).view(torch.bfloat16).cuda()


@pytest.mark.parametrize("b", [1, 3, 4])
def test_exact_ties(b):
    for g in GROUPS:
        W = _tie_matrix(16, 8 * g, g, b, seed=b * 10 + g)
        check_bits(W, g, (b, b, 2), where=f"ties b{b} g{g}")


def test_forced_exact_path():
    W = workloads.generate(96, 512, 4, "t3_rowout", "cuda")
    binding.rrq_set_debug_flags(1)
    try:
        for bits in ((1, 3), (4, 2, 1, 3)):
            check_bits(W, 128, bits, where=f"forced exact {bits}")
    finally:
        binding.rrq_set_debug_flags(0)


def test_batch_across_launches():
    rng = np.random.default_rng(21)
    shapes = [(int(rng.integers(1, 30)), 128 * int(rng.integers(1, 10))) for _ in range(70)]
    mats = [workloads.generate(r, c, 1500 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    bits = [1, 3, 4]
    pkgs = binding.rrq_quantize_ex(mats, 128, 3, binding.GRID_ASYM, binding.SCALE_F32, bits=bits)
    outs = binding.rrq_reconstruct_ex(pkgs, 3, all_prefixes=True)
    torch.cuda.synchronize()
    for i, (W, p) in enumerate(zip(mats, pkgs)):
        rc, rs, rz = oracle.quantize_bits(bf16_bits(W), 128, bits)
        for k in range(3):
            assert np.array_equal(p.codes[k].cpu().numpy(), rc[k]), f"item {i} stage {k}"
        for k in range(1, 4):
            want = oracle.reconstruct_bits(rc, rs, rz, W.shape[0], W.shape[1], 128, k, bits)
            assert np.array_equal(bf16_bits(outs[i][k - 1]), want), f"item {i} prefix {k}"


def test_unsupported_combinations():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    with pytest.raises(binding.RRQError) as e:   # widths other than 2 on the symmetric grid
        binding.rrq_quantize_ex([W], 128, 2, binding.GRID_SYM, binding.SCALE_F16, bits=[1, 3])
    assert e.value.status == 2
    with pytest.raises(binding.RRQError) as e:   # width 5
        binding.rrq_quantize_ex([W], 128, 2, binding.GRID_ASYM, binding.SCALE_F32, bits=[5, 3])
    assert e.value.status == 1
    # (the base branch and the products take widths: tests/test_gpu_base.py,
    # tests/test_gpu_gemv.py, tests/test_gpu_prefill.py)


@pytest.mark.parametrize("group", GROUPS)
def test_group_pmr(group):
    mats = [workloads.generate(r, c, 7 + i, d, "cuda") for i, (r, c, d) in
            enumerate([(64, 4 * group, "t3_rowout"), (3, 8 * group, "normal"), (1024, 1024, "t3_col0.01")])]
    z = torch.zeros((2, 2 * group), dtype=torch.bfloat16, device="cuda")
    z[0, 5] = -1.5  # a group with one nonzero: pmr = group exactly
    mats.append(z)
    pmrs, stats = binding.rrq_group_pmr(mats, group)
    torch.cuda.synchronize()
    for i, (W, pm, st) in enumerate(zip(mats, pmrs, stats)):
        want = oracle.group_pmr(bf16_bits(W), group)
        got = pm.cpu().numpy().astype(np.float64)
        tol = (group + 2) * 2.0 ** -24 * want + 1e-30
        assert np.all(np.abs(got - want) <= tol), f"matrix {i}: max rel err {np.max(np.abs(got - want) / np.maximum(want, 1e-30))}"
        s = st.cpu().numpy().astype(np.float64)
        assert abs(s[0] - want.max()) <= (group + 2) * 2.0 ** -24 * want.max() + 1e-30
        assert abs(s[1] - want.mean()) <= (group + 4) * 2.0 ** -24 * want.max() + 1e-30
    assert pmrs[3].cpu().tolist()[:2] == [float(group), 0.0] and pmrs[3].cpu().tolist()[2:] == [0.0, 0.0]
