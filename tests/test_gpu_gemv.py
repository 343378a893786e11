"""GPU parity for the stage-wise product (rrq_gemv, Appendix C): Y = A W~^T
from the package alone, against the oracle's binary64 product of the same
binary32 prefix weights W~.

Two forms, two bounds.  Groups of 64 and more with 2-bit stages take the
per-group factored form on the tensor cores (gemv_mma_kernel.cuh): per group
and stage s D + lo S (or s (D - 2 S)) with D the codes' product with the
activations; it never forms W~, and its distance to the oracle is at most
d * 2^-24 * sum_c sum_k (|lo_k| + 3 s_k) |a_c| (asymmetric; 2 s_k for the
symmetric grid) with d = (k + 1) + g/16 + 8 + 2k groups + 18 (the kernel's
header derives it).  Packages whose levels and activations are small
integers make every sum exact: those must match bit for bit.

The prefix-weight form (groups of 32, per-stage widths) keeps this bound:
every product W~ a is exact inside
its fma and every partial sum is rounded once; a lane sums its lc columns of
each 32 lc-column window (lc = 128 at k = 1 and at k = 2 with batch <= 2,
else 64, never more than the group) into two accumulators (lc/2 columns each, windows in turn), then
adds the two and the warp adds 32 lanes in 5 butterfly steps, so no term
passes through more than d = 64 ceil(cols/4096) + 8 roundings and
|Y - exact| <= d * 2^-24 * sum_c |W~ a| (first order).  sum_c |W~ a| is
bounded with the bf16 reconstruction: |W~| <= |bf16(W~)| (1 + 2^-8)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bands_intact, bf16_bits, guarded_outputs

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


def _depth(cols):
    """Roundings a term of a row of `cols` columns passes through at most."""
    return 64 * -(-cols // 4096) + 8


def _host_pkg(pkg, rows_idx=None):
    """Package arrays on the host, optionally only the given rows."""
    torch.cuda.synchronize()
    g, cols = pkg.group, pkg.cols
    f16 = pkg.scale_type == binding.SCALE_F16

    def take(t, per_row):
        a = t.view(torch.int16).cpu().numpy().view(np.uint16) if (f16 and t.dtype == torch.float16) \
            else t.cpu().numpy()
        if rows_idx is None:
            return a
        return a.reshape(-1, per_row)[rows_idx].reshape(-1)
    codes = [take(c, cols // 4) for c in pkg.codes]
    scales = [take(s, cols // g) for s in pkg.scales]
    zeros = [take(z, cols // g) for z in pkg.zeros] if pkg.zeros else None
    return codes, scales, zeros


def factored(pkg) -> bool:
    """The package takes the tensor-core form (2-bit stages, groups >= 64)."""
    return pkg.group >= 64 and all(b == 2 for b in pkg.bits[:pkg.n_stages])


def _depth_factored(cols, group, k):
    return (k + 1) + group // 16 + 8 + 2 * k * (cols // group) + 18


def _level_bound(scales, zeros, nr, cols, group, k, sym, f16):
    """Per row and group: sum over the first k stages of |lo| + 3 s (2 s for
    the symmetric grid), float64 [rows, groups]."""
    T = np.zeros((nr, cols // group))
    for i in range(k):
        sc = scales[i].view(np.float16) if f16 else scales[i].view(np.float32)
        sc = np.abs(sc.astype(np.float64)).reshape(nr, -1)
        T += 2 * sc if sym else 3 * sc + np.abs(zeros[i].astype(np.float64)).reshape(nr, -1)
    return T


def _check(pkg, A, Y, k, rows_idx=None, where=""):
    """Y (GPU, float32 [batch, rows]) against the oracle on the given rows."""
    sym, f16 = pkg.grid == binding.GRID_SYM, pkg.scale_type == binding.SCALE_F16
    codes, scales, zeros = _host_pkg(pkg, rows_idx)
    nr = pkg.rows if rows_idx is None else len(rows_idx)
    Ab = bf16_bits(A)
    want = oracle.gemv(codes, scales, zeros, nr, pkg.cols, pkg.group, k, Ab, sym, f16)
    Af = np.abs((Ab.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    if factored(pkg):
        T = _level_bound(scales, zeros, nr, pkg.cols, pkg.group, k, sym, f16)
        Ag = Af.reshape(Af.shape[0], -1, pkg.group).sum(axis=2)
        tol = _depth_factored(pkg.cols, pkg.group, k) * 2.0 ** -24 * (Ag @ T.T) + 1e-30
    else:
        if sym:
            rec = oracle.reconstruct_sym(codes, scales, nr, pkg.cols, pkg.group, k, f16)
        else:
            rec = oracle.reconstruct(codes, scales, zeros, nr, pkg.cols, pkg.group, k)
        recf = np.abs((rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
        d = _depth(pkg.cols)
        tol = d * 2.0 ** -24 * (Af @ recf.T) * (1 + 2.0 ** -8) + 1e-30
    got = Y.cpu().numpy().astype(np.float64)
    if rows_idx is not None:
        got = got[:, rows_idx]
    err = np.abs(got - want)
    bad = np.argwhere(err > tol)
    assert bad.size == 0, (f"{where}: {len(bad)} outputs beyond the bound, first {tuple(bad[0])}: "
                           f"gpu {got[tuple(bad[0])]!r} oracle {want[tuple(bad[0])]!r} tol {tol[tuple(bad[0])]!r}")


def _acts(batch, cols, seed, dev="cuda"):
    g = torch.Generator(device=dev).manual_seed(seed)
    return torch.randn((batch, cols), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("batch", [1, 3, 8])
def test_formats_groups_batches(batch, group, fmt):
    rows, cols = 45, 9 * group  # cols not a multiple of 1024 for g <= 64: ragged chunks
    W = workloads.generate(rows, cols, 70 + group, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, 4, *fmt)
    A = _acts(batch, cols, seed=batch * 100 + group)
    for k in (1, 2, 3, 4):
        (Y,) = binding.rrq_gemv([pkg], [A], k)
        _check(pkg, A, Y, k, where=f"{fmt} g{group} B{batch} k{k}")


@pytest.mark.parametrize("shape", [(1, 32), (3, 96), (7, 2304), (33, 1024 + 32), (5, 12288), (2049, 128)])
def test_shapes(shape):
    rows, cols = shape
    g = 32 if cols % 64 else 128 if cols % 128 == 0 else 64
    W = workloads.generate(rows, cols, rows + cols, "t3", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], g, 4, binding.GRID_ASYM, binding.SCALE_F32)
    A = _acts(2, cols, seed=rows)
    for k in (1, 4):
        (Y,) = binding.rrq_gemv([pkg], [A], k)
        _check(pkg, A, Y, k, where=f"{shape} k{k}")


def test_deterministic_and_matches_asym_original_package():
    """Two calls give identical bits; a package built by rrq_quantize (the
    asymmetric original call) is read the same way."""
    W = workloads.generate(300, 4096, 3, "t3_rowout", "cuda")
    pkg = binding.rrq_quantize(W, 128, 4)
    A = _acts(4, 4096, seed=5)
    Y1 = binding.rrq_gemv([pkg], [A], 4)[0]
    Y2 = binding.rrq_gemv([pkg], [A], 4)[0]
    torch.cuda.synchronize()
    assert torch.equal(Y1.view(torch.int32), Y2.view(torch.int32))
    _check(pkg, A, Y1, 4, where="asym original")


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", [64, 128, 256])
def test_integer_packages_exact(group, fmt):
    """Levels and activations that are small integers make every product and
    sum exact in binary32 (and in the tensor cores): the factored form must
    equal the oracle's product bit for bit, for every prefix and batch."""
    rows, cols = 37, 6 * group
    sym, f16 = fmt[0] == binding.GRID_SYM, fmt[1] == binding.SCALE_F16
    pkg = binding.Package.empty(rows, cols, group, 4, grid=fmt[0], scale_type=fmt[1])
    gen = torch.Generator(device="cuda").manual_seed(group + 7 * fmt[0] + 3 * fmt[1])
    n = rows * cols
    for i in range(4):
        pkg.codes[i].copy_(torch.randint(0, 256, (n // 4,), generator=gen, device="cuda", dtype=torch.int32).to(torch.uint8))
        sc = torch.randint(1, 4, (n // group,), generator=gen, device="cuda").to(torch.float32)
        pkg.scales[i].copy_(sc.to(pkg.scales[i].dtype))
        if not sym:
            pkg.zeros[i].copy_(torch.randint(-6, 3, (n // group,), generator=gen, device="cuda").to(torch.float32))
    for batch in (1, 5, 8):
        A = torch.randint(-3, 4, (batch, cols), generator=gen, device="cuda").to(torch.bfloat16)
        codes, scales, zeros = _host_pkg(pkg)
        for k in (1, 2, 3, 4):
            (Y,) = binding.rrq_gemv([pkg], [A], k)
            want = oracle.gemv(codes, scales, zeros, rows, cols, group, k, bf16_bits(A), sym, f16)
            got = Y.cpu().numpy().astype(np.float64)
            assert np.array_equal(got, want), f"g{group} {fmt} B{batch} k{k}: {int((got != want).sum())} differ"


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", [64, 128, 256])
def test_activation_scales(group, fmt):
    """The tensor-core form works in a domain scaled per activation row by a
    power of two taken from the row's largest exponent: a row times 2^j gives
    outputs times exactly 2^j (the same roundings), for rows of very different
    magnitudes in one call; a row of zeros gives zeros; a row whose columns
    span 2^-60 .. 2^60 stays within the bound."""
    rows, cols = 40, 8 * group
    W = workloads.generate(rows, cols, 90 + group, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, 4, *fmt)
    gen = torch.Generator(device="cuda").manual_seed(group + fmt[1])
    z = torch.randn((1, cols), generator=gen, device="cuda")
    base = (torch.sign(z) * (0.5 + z.abs())).to(torch.bfloat16)  # |a| >= 0.5: no row is scaled into subnormals
    js = [0, -100, 100, -60, 60]
    ex = torch.randint(-60, 61, (1, cols), generator=gen, device="cuda").to(torch.float32)
    mixed = (base.float() * torch.exp2(ex)).to(torch.bfloat16)
    A = torch.cat([(base.float() * 2.0 ** j).to(torch.bfloat16) for j in js]
                  + [torch.zeros((1, cols), device="cuda", dtype=torch.bfloat16), mixed])
    for k in (1, 2, 3, 4):
        (Y,) = binding.rrq_gemv([pkg], [A], k)
        for i, j in enumerate(js):
            assert torch.equal(Y[i], Y[0] * 2.0 ** j), f"g{group} {fmt} k{k}: row scaled by 2^{j}"
        assert torch.count_nonzero(Y[len(js)]) == 0
        _check(pkg, A, Y, k, where=f"g{group} {fmt} k{k} scaled rows")


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
def test_one_warp_per_block(fmt):
    """A launch with at least 16 blocks of 16 rows in every CTA takes one warp
    per block (the form the whole stack takes); smaller launches share each
    block among a group of warps.  Both against the oracle on every row."""
    rows, cols, group = 40960, 512, 128  # 2560 blocks over at most 152 CTAs
    W = workloads.generate(rows, cols, 91, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, 4, *fmt)
    for batch in (1, 5):
        A = _acts(batch, cols, seed=batch + 17)
        for k in (1, 4):
            (Y,) = binding.rrq_gemv([pkg], [A], k)
            _check(pkg, A, Y, k, where=f"{fmt} B{batch} k{k}")


def test_batch_across_launches():
    rng = np.random.default_rng(12)
    shapes = [(int(rng.integers(1, 40)), 128 * int(rng.integers(1, 20))) for _ in range(70)]
    mats = [workloads.generate(r, c, 1200 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_ex(mats, 128, 4, binding.GRID_SYM, binding.SCALE_F16)
    acts = [_acts(2, c, seed=i) for i, (r, c) in enumerate(shapes)]
    ys = binding.rrq_gemv(pkgs, acts, 3)
    for i, (p, A, Y) in enumerate(zip(pkgs, acts, ys)):
        _check(p, A, Y, 3, where=f"item {i}")


def test_qwen3_8b_layer_sampled_rows():
    """A full-size Qwen3-8B-shaped layer (7 matrices, one call) at batch 1,
    every prefix; 64 sampled rows of every matrix against the oracle."""
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    acts = [_acts(1, sp.cols, seed=50 + i) for i, sp in enumerate(specs)]
    for k in (1, 2, 3, 4):
        ys = binding.rrq_gemv(pkgs, acts, k)
        for i, (sp, p, A, Y) in enumerate(zip(specs, pkgs, acts, ys)):
            rng = np.random.default_rng(i * 10 + k)
            idx = np.unique(np.concatenate([[0, sp.rows - 1], rng.integers(0, sp.rows, 62)]))
            _check(p, A, Y, k, rows_idx=idx, where=f"{sp.name} k{k}")


@pytest.mark.parametrize("group", [32, 128])
@pytest.mark.parametrize("bits", [(1, 3), (3, 1), (4, 2, 1), (2, 4), (1, 1, 1, 1), (4, 4)],
                         ids=lambda b: "+".join(map(str, b)))
@pytest.mark.parametrize("batch", [1, 5])
def test_widths(batch, bits, group):
    """Packages with per-stage widths: every prefix against the oracle's
    decode form (binary32 prefix weights) within the kernel's summation
    bound (the same tree as the 2-bit formats)."""
    rows, cols = 45, 9 * group
    W = workloads.generate(rows, cols, 95 + sum(bits), "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, len(bits), binding.GRID_ASYM, binding.SCALE_F32, bits=bits)
    A = _acts(batch, cols, seed=batch + group)
    torch.cuda.synchronize()
    codes = [c.cpu().numpy() for c in pkg.codes]
    scales = [x.cpu().numpy() for x in pkg.scales]
    zeros = [x.cpu().numpy() for x in pkg.zeros]
    Ab = bf16_bits(A)
    Af = np.abs((Ab.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    for k in range(1, len(bits) + 1):
        (Y,) = binding.rrq_gemv([pkg], [A], k)
        want = oracle.product_bits(codes, scales, zeros, rows, cols, group, k, bits, Ab, False)
        rec = oracle.reconstruct_bits(codes, scales, zeros, rows, cols, group, k, bits)
        recf = np.abs((rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
        d = _depth(cols)
        tol = d * 2.0 ** -24 * (Af @ recf.T) * (1 + 2.0 ** -8) + 1e-30
        err = np.abs(Y.cpu().numpy().astype(np.float64) - want)
        assert not np.any(err > tol), f"{bits} g{group} B{batch} k{k}: {int((err > tol).sum())} outputs beyond the bound"


def test_widest_rows_and_batch_split():
    """The widest supported rows (RRQ_MAX_GEMV_COLS columns: one activation
    row fits a launch's shared memory) and a batch of 8 at 28672 columns (two
    activation rows per launch in the tensor-core form at group 128: four
    launches over the same package)."""
    for rows, cols, batch in ((3, 57344, 1), (5, 28672, 8)):
        W = workloads.generate(rows, cols, cols + batch, "t3_rowout", "cuda")
        (pkg,) = binding.rrq_quantize_ex([W], 128, 4, binding.GRID_ASYM, binding.SCALE_F32)
        A = _acts(batch, cols, seed=rows)
        for k in (1, 4):
            (Y,) = binding.rrq_gemv([pkg], [A], k)
            _check(pkg, A, Y, k, where=f"{rows}x{cols} B{batch} k{k}")


def test_mixed_widths_batch_8():
    """One call at batch 8 over matrices of 4096, 12288, 28672 and 57344
    columns, which hold different numbers of activation rows per launch (8,
    5, 2 and 1 in the tensor-core form at group 128): each width class is
    launched on its own share of the batch, in any order of the items."""
    shapes = [(5, 28672), (7, 4096), (3, 57344), (17, 12288), (2, 4096)]
    mats = [workloads.generate(r, c, 300 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_ex(mats, 128, 2, binding.GRID_ASYM, binding.SCALE_F32)
    acts = [_acts(8, c, seed=40 + i) for i, (r, c) in enumerate(shapes)]
    for k in (1, 2):
        ys = binding.rrq_gemv(pkgs, acts, k)
        for i, (p, A, Y) in enumerate(zip(pkgs, acts, ys)):
            _check(p, A, Y, k, where=f"item {i} {shapes[i]} k{k}")


def test_too_wide():
    cols = 57344 + 128
    W = workloads.generate(1, cols, 9, "normal", "cuda")
    pkg = binding.rrq_quantize(W, 128, 1)
    A = _acts(1, cols, seed=3)
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_gemv([pkg], [A], 1)
    assert e.value.status == 2


def test_errors():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    pkg = binding.rrq_quantize(W, 128, 2)
    A = _acts(9, 256, seed=1)
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_gemv([pkg], [A], 1)
    assert e.value.status == 1
    with pytest.raises(ValueError):
        binding.rrq_gemv([pkg], [A[:2]], 3)
    A2 = _acts(2, 256, seed=2)
    Yover = A2.view(torch.float32).reshape(-1)[:16].view(2, 8)  # Y over the activations
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_gemv([pkg], [A2], 1, ys=[Yover])
    assert e.value.status == 1


def test_guard_bands_untouched():
    """Outputs inside 4 KiB sentinel bands: ragged shapes (rows not a
    multiple of 16, a group of 32, a partial window) at batches 1 and 3 and
    every k write inside their [batch, rows] only."""
    shapes = [(45, 384), (3, 4096 + 128), (17, 1152)]
    mats = [workloads.generate(r, c, 500 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    for group in (32, 128):
        pkgs = [binding.rrq_quantize_ex([W], group, 4, binding.GRID_ASYM, binding.SCALE_F32)[0] for W in mats]
        for batch in (1, 3):
            acts = [_acts(batch, c, seed=60 + i) for i, (r, c) in enumerate(shapes)]
            for k in (1, 4):
                bufs, ys, guard = guarded_outputs(shapes, batch)
                binding.rrq_gemv(pkgs, acts, k, ys)
                assert bands_intact(bufs, guard), f"g{group} batch {batch} k {k}: a sentinel band changed"
                for i, (p, A, Y) in enumerate(zip(pkgs, acts, ys)):
                    _check(p, A, Y, k, where=f"guarded item {i} g{group} B{batch} k{k}")
