"""GPU parity for the symmetric package (implicit zero-point 2, levels
(Q-2)s, s = 2 max|x| / 3; the paper's "symmetric" configuration with 16-bit
scales, Table 4 and Appendix G) through rrq_quantize_ex /
rrq_reconstruct_ex: codes and binary32 or binary16 scales bit for bit, and
every bf16 prefix with 0 ULP, against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import (bf16_bits, check_full, check_full_sym, check_sampled_sym, scales_host,
                         gpu_package_host, sample_groups)

pytestmark = pytest.mark.gpu

GROUPS = (32, 64, 128, 256)
SCALES = (False, True)  # binary16 scales?


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)
    yield
    binding.rrq_set_debug_flags(0)


def test_single_4096_f16():
    W = workloads.generate(4096, 4096, 0, "normal", "cuda")
    check_full_sym(W, 128, 4, True, where="sym f16 4096")


@pytest.mark.parametrize("f16", SCALES)
@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("dist", ["normal", "t3", "t3_rowout", "t3_col0.01"])
def test_groups_and_distributions(dist, group, f16):
    W = workloads.generate(333, 5 * group, 29 + group, dist, "cuda")
    check_full_sym(W, group, 4, f16, where=f"sym {dist} g{group} f16={f16}")


@pytest.mark.parametrize("f16", SCALES)
@pytest.mark.parametrize("n_stages", [1, 2, 3])
def test_fewer_stages(n_stages, f16):
    for g in GROUPS:
        W = workloads.generate(64, 4 * g, 6, "t3_rowout", "cuda")
        check_full_sym(W, g, n_stages, f16, where=f"sym S={n_stages} g{g}")


@pytest.mark.parametrize("f16", SCALES)
@pytest.mark.parametrize("shape", [(1, 32), (3, 32), (31, 32), (1, 64), (1, 128), (1, 256),
                                   (3, 256), (1, 1024 + 32), (7, 2304), (2049, 128)])
def test_small_and_ragged_shapes(shape, f16):
    """Including odd group counts: the last binary16 scale of an array sits in
    a 4-byte word of which only 2 bytes belong to the array."""
    rows, cols = shape
    for g in GROUPS:
        if cols % g:
            continue
        W = workloads.generate(rows, cols, rows * 11 + cols, "t3", "cuda")
        check_full_sym(W, g, 4, f16, where=f"sym {shape} g{g} f16={f16}")


def _sym_edge_matrix(rows, cols, group, seed, huge: bool):
    """Groups of: Gaussian, constant, signed zeros, values on the symmetric
    grid with exact ties, bf16 subnormals, tiny magnitudes whose binary16
    scale is subnormal or rounds to 0, a single nonzero, and (binary32 scales
    only) huge magnitudes."""
    rng = np.random.default_rng(seed)
    n_groups = rows * cols // group
    out = np.empty((n_groups, group), np.uint16)

    def bf16(x):
        u = np.asarray(x, np.float32).view(np.uint32)
        return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)

    for gi in range(n_groups):
        kind = gi % 9
        if kind == 0:
            out[gi] = bf16(rng.normal(0, 0.02, group))
        elif kind == 1:
            out[gi] = bf16(np.full(group, rng.normal(0, 1)))
        elif kind == 2:
            out[gi] = rng.choice(np.array([0x0000, 0x8000], np.uint16), group)
        elif kind == 3:  # m/4 * s with s = 2^e, amax = 1.5 s: exact ties at +-0.5, +-1.5
            e = int(rng.integers(-8, 2))
            m = rng.integers(-6, 7, group)
            m[0] = 6 if rng.random() < 0.5 else -6
            out[gi] = bf16(m * 2.0 ** (e - 2))
        elif kind == 4:
            out[gi] = rng.integers(0, 0x80, group).astype(np.uint16) | \
                (rng.integers(0, 2, group).astype(np.uint16) << 15)
        elif kind == 5:  # binary16 scale in the subnormal range or rounding to 0
            out[gi] = bf16(rng.normal(0, 2.0 ** -float(rng.integers(14, 30)), group))
        elif kind == 6:
            v = np.zeros(group)
            v[rng.integers(0, group)] = rng.normal(0, 0.1)
            out[gi] = bf16(v)
        elif kind == 7 and huge:
            out[gi] = bf16(rng.normal(0, 1e30, group))
        else:
            out[gi] = bf16(rng.standard_t(3, group) * 0.02)
    W = torch.from_numpy(out.reshape(rows, cols).view(np.int16)).view(torch.bfloat16)
    return W.cuda()


@pytest.mark.parametrize("f16", SCALES)
@pytest.mark.parametrize("group", GROUPS)
def test_edge_case_groups(group, f16):
    W = _sym_edge_matrix(40, 9 * group, group, seed=group + 5, huge=not f16)
    check_full_sym(W, group, 4, f16, where=f"sym edge g{group} f16={f16}")


@pytest.mark.parametrize("f16", SCALES)
@pytest.mark.parametrize("group", GROUPS)
def test_forced_exact_path_matches(group, f16):
    W = _sym_edge_matrix(16, 9 * group, group, seed=200 + group, huge=not f16)
    binding.rrq_set_debug_flags(1)
    try:
        check_full_sym(W, group, 4, f16, where=f"sym forced-exact g{group} f16={f16}")
    finally:
        binding.rrq_set_debug_flags(0)


def test_batch_across_launches_f16():
    """70 matrices of mixed shapes (two launches of the 64-matrix kernels)."""
    rng = np.random.default_rng(4)
    shapes = [(int(rng.integers(1, 40)), 128 * int(rng.integers(1, 12))) for _ in range(70)]
    mats = [workloads.generate(r, c, 500 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_ex(mats, 128, 4, binding.GRID_SYM, binding.SCALE_F16)
    outs = binding.rrq_reconstruct_ex(pkgs, 4, all_prefixes=True)
    one = binding.rrq_reconstruct_ex(pkgs, 2)
    torch.cuda.synchronize()
    for i, (W, pkg) in enumerate(zip(mats, pkgs)):
        rc, rs = oracle.quantize_sym(bf16_bits(W), 128, 4, True)
        gs = scales_host(pkg)
        for k in range(4):
            assert np.array_equal(pkg.codes[k].cpu().numpy(), rc[k]), f"item {i} stage {k} codes"
            assert np.array_equal(gs[k], rs[k]), f"item {i} stage {k} scales"
        for k in range(1, 5):
            want = oracle.reconstruct_sym(rc, rs, W.shape[0], W.shape[1], 128, k, True)
            assert np.array_equal(bf16_bits(outs[i][k - 1]), want), f"item {i} prefix {k}"
        assert np.array_equal(bf16_bits(one[i][0]),
                              oracle.reconstruct_sym(rc, rs, W.shape[0], W.shape[1], 128, 2, True))


def test_asym_through_ex_equals_original_calls():
    """rrq_quantize_ex / rrq_reconstruct_ex with the asymmetric grid and
    binary32 scales give the same bits as rrq_quantize / rrq_reconstruct."""
    W = workloads.generate(257, 640, 8, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], 128, 4, binding.GRID_ASYM, binding.SCALE_F32)
    ref_pkg = check_full(W, 128, 4, where="asym via original calls")
    a, b = gpu_package_host(pkg), gpu_package_host(ref_pkg)
    for x, y in zip(a, b):
        for u, v in zip(x, y):
            assert np.array_equal(u.view(np.uint8), v.view(np.uint8))
    outs = binding.rrq_reconstruct_ex([pkg], 4, all_prefixes=True)[0]
    for k in (1, 2, 3, 4):
        assert torch.equal(outs[k - 1].view(torch.int16), binding.rrq_reconstruct(ref_pkg, k).view(torch.int16))


def test_guard_bands_f16_odd_groups():
    """binary16 scale arrays with an odd number of groups, each between 4 KiB
    sentinel bands: neither kernel writes outside its outputs, and the
    reconstruction reads only the array's own 2-byte tail."""
    rows, cols, g, S = 7, 3 * 32, 32, 4  # 21 groups
    n = rows * cols
    guard = 4096
    W = workloads.generate(rows, cols, 12, "t3_rowout", "cuda")

    def guarded(nbytes, fill=0xA5):
        buf = torch.full((nbytes + 2 * guard,), fill, dtype=torch.uint8, device="cuda")
        return buf, buf[guard:guard + nbytes]

    bufs, codes, scales = [], [], []
    for _ in range(S):
        b, c = guarded(n // 4); bufs.append(b); codes.append(c)
        b, s = guarded(2 * (n // g)); bufs.append(b); scales.append(s.view(torch.float16))
    pkg = binding.Package(codes, scales, [], rows, cols, g, S, binding.GRID_SYM, binding.SCALE_F16)
    binding.rrq_quantize_ex([W], g, S, binding.GRID_SYM, binding.SCALE_F16, pkgs=[pkg])
    ob, o = guarded(2 * n)
    binding.rrq_reconstruct_ex([pkg], 4, outs=[[o.view(torch.bfloat16).view(rows, cols)]])
    torch.cuda.synchronize()
    for b in bufs + [ob]:
        h = b.cpu().numpy()
        assert (h[:guard] == 0xA5).all() and (h[-guard:] == 0xA5).all()
    rc, rs = oracle.quantize_sym(bf16_bits(W), g, S, True)
    want = oracle.reconstruct_sym(rc, rs, rows, cols, g, 4, True)
    assert np.array_equal(bf16_bits(o.view(torch.bfloat16).view(rows, cols)), want)


def test_format_errors():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize_ex([W], 128, 4, binding.GRID_ASYM, binding.SCALE_F16)
    assert e.value.status == 2
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize_ex([W], 128, 4, 7, binding.SCALE_F16)
    assert e.value.status == 1
    (pkg,) = binding.rrq_quantize_ex([W], 128, 2)
    with pytest.raises(ValueError):
        binding.rrq_reconstruct_ex([pkg], 3)


def test_qwen3_8b_layer_f16_sampled():
    """One full-size Qwen3-8B-shaped layer (7 matrices) in one batched call,
    sampled groups of every matrix and every prefix against the oracle."""
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = binding.rrq_quantize_ex(mats, 128, 4, binding.GRID_SYM, binding.SCALE_F16)
    outs = binding.rrq_reconstruct_ex(pkgs, 4, all_prefixes=True)
    torch.cuda.synchronize()
    for i, (sp, W, pkg) in enumerate(zip(specs, mats, pkgs)):
        idx = sample_groups(sp.numel // 128, 3000, seed=700 + i)
        check_sampled_sym(W, pkg, idx, outs[i], where=sp.name)
