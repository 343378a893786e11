"""GPU parity for Algorithm 1 with a base checkpoint (rrq_quantize_from_base):
stage 0 of the package is given -- here random codes, scales and zeros, i.e.
a base that round-to-nearest would not produce, with extreme scales mixed in
-- and stages 1.. must equal the CPU oracle's bit for bit, for every format;
given the base the build itself computes, the two branches of Algorithm 1
must agree."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bf16_bits, sample_groups

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


def _random_base(pkg, seed, extremes=True):
    """Fill stage 0 of pkg with random codes, positive scales (a few zero,
    tiny or huge ones) and, for the asymmetric grid, negative zeros."""
    rng = np.random.default_rng(seed)
    n_groups = pkg.scales[0].numel()
    pkg.codes[0].copy_(torch.from_numpy(rng.integers(0, 256, pkg.codes[0].numel()).astype(np.uint8)))
    if pkg.scale_type == binding.SCALE_F16:
        s = rng.uniform(2.0 ** -12, 0.05, n_groups).astype(np.float16)
        if extremes:
            s[::17] = np.float16(0)
            s[5::23] = np.float16(2.0 ** -24) * rng.integers(1, 1023, s[5::23].size).astype(np.float16)
        pkg.scales[0].copy_(torch.from_numpy(s))
    else:
        s = rng.uniform(1e-3, 0.05, n_groups).astype(np.float32)
        if extremes:
            s[::17] = 0.0
            s[5::23] = np.float32(1e-40)   # subnormal
            s[7::29] = np.float32(3e31)    # beyond 2^100
        pkg.scales[0].copy_(torch.from_numpy(s))
    if pkg.grid == binding.GRID_ASYM:
        z = rng.uniform(-0.1, 0.0, n_groups).astype(np.float32)
        pkg.zeros[0].copy_(torch.from_numpy(z))


def _host(pkg):
    torch.cuda.synchronize()
    f16 = pkg.scale_type == binding.SCALE_F16
    codes = [c.cpu().numpy() for c in pkg.codes]
    scales = [s.view(torch.int16).cpu().numpy().view(np.uint16) if f16 else s.cpu().numpy() for s in pkg.scales]
    zeros = [z.cpu().numpy() for z in pkg.zeros] if pkg.zeros else None
    return codes, scales, zeros


def _check(W, pkg, where):
    """Package of pkg (stage 0 given) against the oracle's, and every prefix."""
    rows, cols = W.shape
    g, S = pkg.group, pkg.n_stages
    sym, f16 = pkg.grid == binding.GRID_SYM, pkg.scale_type == binding.SCALE_F16
    gc, gs, gz = _host(pkg)
    base = (gc[0], gs[0], gz[0] if gz else None)
    rc, rs, rz = oracle.quantize_from_base(bf16_bits(W), base, g, S, sym, f16)
    for k in range(S):
        assert np.array_equal(gc[k], rc[k]), f"{where} stage {k} codes"
        assert np.array_equal(gs[k].view(np.uint8), rs[k].view(np.uint8)), f"{where} stage {k} scales"
        if not sym:
            assert np.array_equal(gz[k].view(np.uint32), rz[k].view(np.uint32)), f"{where} stage {k} zeros"
    outs = binding.rrq_reconstruct_ex([pkg], S, all_prefixes=True)[0]
    torch.cuda.synchronize()
    for k in range(1, S + 1):
        want = oracle.reconstruct_sym(rc, rs, rows, cols, g, k, f16) if sym else \
            oracle.reconstruct(rc, rs, rz, rows, cols, g, k)
        assert np.array_equal(bf16_bits(outs[k - 1]), want), f"{where} prefix {k}"


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("dist", ["normal", "t3_rowout"])
def test_random_base(dist, group, fmt):
    W = workloads.generate(133, 5 * group, 41 + group, dist, "cuda")
    (pkg,) = [binding.Package.empty(133, 5 * group, group, 4, W.device, *fmt)]
    _random_base(pkg, seed=group)
    binding.rrq_quantize_from_base([W], [pkg])
    _check(W, pkg, f"{dist} g{group} {fmt}")


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
def test_branches_agree_given_the_rtn_base(fmt):
    """Algorithm 1: starting from the base the build computes itself gives
    the package of the build without a checkpoint, bit for bit."""
    W = workloads.generate(257, 1024, 5, "t3_rowout", "cuda")
    (ref,) = binding.rrq_quantize_ex([W], 128, 4, *fmt)
    pkg = binding.Package.empty(257, 1024, 128, 4, W.device, *fmt)
    pkg.codes[0].copy_(ref.codes[0])
    pkg.scales[0].copy_(ref.scales[0])
    if pkg.zeros:
        pkg.zeros[0].copy_(ref.zeros[0])
    binding.rrq_quantize_from_base([W], [pkg])
    torch.cuda.synchronize()
    for k in range(4):
        assert torch.equal(pkg.codes[k], ref.codes[k])
        assert torch.equal(pkg.scales[k].view(torch.int16 if pkg.scale_type else torch.int32),
                           ref.scales[k].view(torch.int16 if pkg.scale_type else torch.int32))
        if pkg.zeros:
            assert torch.equal(pkg.zeros[k].view(torch.int32), ref.zeros[k].view(torch.int32))


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("shape", [(1, 32), (3, 32), (31, 32), (1, 1024 + 32), (7, 2304), (2049, 128)])
def test_ragged_shapes_two_stages(shape, fmt):
    rows, cols = shape
    for g in GROUPS:
        if cols % g:
            continue
        for S in (2, 4):
            W = workloads.generate(rows, cols, rows + cols + S, "t3", "cuda")
            pkg = binding.Package.empty(rows, cols, g, S, W.device, *fmt)
            _random_base(pkg, seed=rows * 3 + g + S)
            binding.rrq_quantize_from_base([W], [pkg])
            _check(W, pkg, f"{shape} g{g} S{S} {fmt}")


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
def test_forced_exact_path(fmt):
    W = workloads.generate(96, 512, 3, "t3_rowout", "cuda")
    pkg = binding.Package.empty(96, 512, 128, 4, W.device, *fmt)
    _random_base(pkg, seed=9)
    binding.rrq_set_debug_flags(1)
    try:
        binding.rrq_quantize_from_base([W], [pkg])
        _check(W, pkg, f"forced exact {fmt}")
    finally:
        binding.rrq_set_debug_flags(0)


def test_batch_across_launches():
    rng = np.random.default_rng(8)
    shapes = [(int(rng.integers(1, 40)), 128 * int(rng.integers(1, 12))) for _ in range(70)]
    mats = [workloads.generate(r, c, 900 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    fmt = (binding.GRID_SYM, binding.SCALE_F16)
    pkgs = [binding.Package.empty(r, c, 128, 4, mats[0].device, *fmt) for r, c in shapes]
    for i, p in enumerate(pkgs):
        _random_base(p, seed=1000 + i)
    binding.rrq_quantize_from_base(mats, pkgs)
    for i, (W, p) in enumerate(zip(mats, pkgs)):
        _check(W, p, f"batch item {i}")


BIT_SPLITS = [(1, 3), (3, 1), (4, 2, 1), (2, 4, 2, 1)]


def _check_bits(W, pkg, bits, where):
    """Stages 1.. of pkg against the oracle's base branch with widths, given
    the package's own stage 0."""
    codes, scales, zeros = _host(pkg)
    rc, rs, rz = oracle.quantize_from_base_bits(bf16_bits(W), (codes[0], scales[0], zeros[0]), pkg.group,
                                                list(bits))
    for k in range(1, len(bits)):
        assert np.array_equal(codes[k], rc[k]), f"{where} stage {k} codes"
        assert np.array_equal(scales[k].view(np.uint32), rs[k].view(np.uint32)), f"{where} stage {k} scales"
        assert np.array_equal(zeros[k].view(np.uint32), rz[k].view(np.uint32)), f"{where} stage {k} zeros"


@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("bits", BIT_SPLITS, ids=lambda b: "+".join(map(str, b)))
def test_widths_random_base(bits, group):
    """Per-stage widths: a random base (random codes, zero, subnormal and
    huge scales) at width bits[0], stages 1.. bit for bit against the oracle."""
    rows, cols = 67, 5 * group
    W = workloads.generate(rows, cols, 40 + group, "t3_rowout", "cuda")
    pkg = binding.Package.empty(rows, cols, group, len(bits), W.device, binding.GRID_ASYM, binding.SCALE_F32,
                                bits=bits)
    _random_base(pkg, seed=group + 10 * len(bits))
    binding.rrq_quantize_from_base([W], [pkg])
    _check_bits(W, pkg, bits, where=f"{bits} g{group}")
    assert binding.rrq_get_device_status() == 0


@pytest.mark.parametrize("bits", BIT_SPLITS, ids=lambda b: "+".join(map(str, b)))
def test_widths_branches_agree(bits):
    """Given the width package's own RTN stage 0, the base branch rebuilds the
    same package on the device."""
    W = workloads.generate(200, 1024, 55, "t3_rowout", "cuda")
    (full,) = binding.rrq_quantize_ex([W], 128, len(bits), binding.GRID_ASYM, binding.SCALE_F32, bits=bits)
    pkg = binding.Package.empty(200, 1024, 128, len(bits), W.device, binding.GRID_ASYM, binding.SCALE_F32, bits=bits)
    pkg.codes[0].copy_(full.codes[0])
    pkg.scales[0].copy_(full.scales[0])
    pkg.zeros[0].copy_(full.zeros[0])
    binding.rrq_quantize_from_base([W], [pkg])
    torch.cuda.synchronize()
    for k in range(len(bits)):
        assert torch.equal(pkg.codes[k], full.codes[k]), f"{bits} stage {k} codes"
        assert torch.equal(pkg.scales[k].view(torch.int32), full.scales[k].view(torch.int32)), f"{bits} stage {k}"
        assert torch.equal(pkg.zeros[k].view(torch.int32), full.zeros[k].view(torch.int32)), f"{bits} stage {k}"


def test_errors():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    pkg = binding.Package.empty(8, 256, 128, 1, W.device, binding.GRID_SYM, binding.SCALE_F16)
    with pytest.raises(binding.RRQError) as e:   # nothing to compute: one stage
        binding.rrq_quantize_from_base([W], [pkg])
    assert e.value.status == 1
    pkg = binding.Package.empty(8, 256, 128, 4, W.device, binding.GRID_ASYM, binding.SCALE_F32)
    pkg.codes[2] = pkg.codes[0]                 # an output over the given base
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize_from_base([W], [pkg])
    assert e.value.status == 1


def test_qwen3_8b_layer_sampled():
    """One full-size Qwen3-8B-shaped layer from random asymmetric bases, one
    batched call; sampled groups against the oracle."""
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = [binding.Package.empty(sp.rows, sp.cols, 128, 4, mats[0].device) for sp in specs]
    for i, p in enumerate(pkgs):
        _random_base(p, seed=60 + i, extremes=False)
    binding.rrq_quantize_from_base(mats, pkgs)
    torch.cuda.synchronize()
    for i, (sp, W, p) in enumerate(zip(specs, mats, pkgs)):
        idx = sample_groups(sp.numel // 128, 2000, seed=800 + i)
        it = torch.from_numpy(idx).cuda()
        Wg = W.reshape(-1, 128).index_select(0, it)
        base = (p.codes[0].view(-1, 32).index_select(0, it).cpu().numpy().reshape(-1),
                p.scales[0].index_select(0, it).cpu().numpy(), p.zeros[0].index_select(0, it).cpu().numpy())
        rc, rs, rz = oracle.quantize_from_base(bf16_bits(Wg), base, 128, 4)
        for k in range(1, 4):
            gc = p.codes[k].view(-1, 32).index_select(0, it).cpu().numpy().reshape(-1)
            assert np.array_equal(gc, rc[k]), f"{sp.name} stage {k} codes"
            assert np.array_equal(p.scales[k].index_select(0, it).cpu().numpy().view(np.uint32),
                                  rs[k].view(np.uint32)), f"{sp.name} stage {k} scales"
            assert np.array_equal(p.zeros[k].index_select(0, it).cpu().numpy().view(np.uint32),
                                  rz[k].view(np.uint32)), f"{sp.name} stage {k} zeros"
