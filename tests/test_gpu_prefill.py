"""GPU parity for the tensor-core prefill product (rrq_prefill, Appendix C's
stage-wise product for many activation rows): Y = A bf16(W~)^T from the
package alone, against the oracle's binary64 product with the bf16 prefix
reconstruction.

Tolerance, from the kernel's arithmetic: the weights the kernel forms are the
bf16 reconstruction bit for bit, and every product of two bf16 values is
exact in binary32.  The tensor cores add the products of one MMA (16 columns)
and the accumulator in binary32; taking each of the cols/16 accumulation
steps as one rounding of at most one unit in the last place (2^-23 relative,
which also covers truncation), |Y - exact| <= (cols/16 + 2) * 2^-23 *
sum_c |a w|.  Packages with integer levels and integer activations make every
partial sum an integer below 2^24, and there the product must be exact."""
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


def _check(pkg, A, Y, k, rows_idx=None, tok_idx=None, where=""):
    """Y (GPU, float32 [tokens, rows]) against the oracle on the given rows
    and tokens."""
    sym, f16 = pkg.grid == binding.GRID_SYM, pkg.scale_type == binding.SCALE_F16
    codes, scales, zeros = _host_pkg(pkg, rows_idx)
    nr = pkg.rows if rows_idx is None else len(rows_idx)
    Ab = bf16_bits(A)
    if tok_idx is not None:
        Ab = Ab[tok_idx]
    want = oracle.prefill(codes, scales, zeros, nr, pkg.cols, pkg.group, k, Ab, sym, f16)
    if sym:
        rec = oracle.reconstruct_sym(codes, scales, nr, pkg.cols, pkg.group, k, f16)
    else:
        rec = oracle.reconstruct(codes, scales, zeros, nr, pkg.cols, pkg.group, k)
    recf = np.abs((rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    Af = np.abs((Ab.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    tol = (pkg.cols / 16 + 2) * 2.0 ** -23 * (Af @ recf.T) + 1e-30
    got = Y.cpu().numpy().astype(np.float64)
    if tok_idx is not None:
        got = got[tok_idx]
    if rows_idx is not None:
        got = got[:, rows_idx]
    err = np.abs(got - want)
    bad = np.argwhere(err > tol)
    assert bad.size == 0, (f"{where}: {len(bad)} outputs beyond the bound, first {tuple(bad[0])}: "
                           f"gpu {got[tuple(bad[0])]!r} oracle {want[tuple(bad[0])]!r} tol {tol[tuple(bad[0])]!r}")
    return float((err / np.maximum(Af @ recf.T, 1e-30)).max())


def _acts(tokens, cols, seed, dev="cuda"):
    g = torch.Generator(device=dev).manual_seed(seed)
    return torch.randn((tokens, cols), generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)


def _status_ok():
    assert binding.rrq_get_device_status() == 0


@pytest.mark.parametrize("fmt", FORMATS, ids=FMT_IDS)
@pytest.mark.parametrize("group", GROUPS)
def test_formats_groups(group, fmt):
    # 200 rows: one full and one ragged row tile; 300 tokens: one full and one
    # ragged token tile; 9 groups of columns: a half stage at the end for g = 32
    rows, cols, tokens = 200, 9 * group, 300
    W = workloads.generate(rows, cols, 80 + group, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, 4, *fmt)
    A = _acts(tokens, cols, seed=group)
    for k in (1, 2, 3, 4):
        (Y,) = binding.rrq_prefill([pkg], [A], k)
        _check(pkg, A, Y, k, where=f"{fmt} g{group} k{k}")
    _status_ok()


def _integer_package(rows, cols, group, seed, dev="cuda"):
    """Asymmetric package with scale 1 and integer zeros in [-3, 3]: every
    level z + Q is an integer, so every prefix weight is one too."""
    rng = np.random.default_rng(seed)
    n = rows * cols
    pkg = binding.Package.empty(rows, cols, group, 4, torch.device(dev))
    for i in range(4):
        pkg.codes[i].copy_(torch.from_numpy(rng.integers(0, 256, n // 4, dtype=np.uint8)))
        pkg.scales[i].fill_(1.0)
        pkg.zeros[i].copy_(torch.from_numpy(rng.integers(-3, 4, n // group).astype(np.float32)))
    return pkg


@pytest.mark.parametrize("shape", [(128, 256, 256), (77, 4096, 130), (300, 1024, 513)])
def test_integer_packages_exact(shape):
    """Integer weights (|w| <= 24) and integer activations (|a| <= 4): every
    partial sum is an integer below 2^24, so Y is exact."""
    rows, cols, tokens = shape
    pkg = _integer_package(rows, cols, 128, seed=rows)
    g = torch.Generator(device="cuda").manual_seed(tokens)
    A = torch.randint(-4, 5, (tokens, cols), generator=g, device="cuda").to(torch.bfloat16)
    codes, scales, zeros = _host_pkg(pkg)
    for k in (1, 4):
        (Y,) = binding.rrq_prefill([pkg], [A], k)
        want = oracle.prefill(codes, scales, zeros, rows, cols, 128, k, bf16_bits(A))
        assert np.array_equal(Y.cpu().numpy().astype(np.float64), want), f"{shape} k{k}"
    _status_ok()


# token tiles of 512: 1 (no cluster), 2 (clusters of 2), 3 and 6 (clusters of
# 4 with idle padding CTAs), 4
@pytest.mark.parametrize("shape", [(1, 32, 1), (3, 96, 7), (129, 4096, 257), (64, 12288, 64), (513, 128, 1000),
                                   (200, 1024, 1100), (77, 2048, 3000), (256, 4096, 2048)])
def test_shapes(shape):
    rows, cols, tokens = shape
    g = 32 if cols % 64 else 128 if cols % 128 == 0 else 64
    W = workloads.generate(rows, cols, rows + cols, "t3", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], g, 4, binding.GRID_ASYM, binding.SCALE_F32)
    A = _acts(tokens, cols, seed=rows)
    for k in (1, 4):
        (Y,) = binding.rrq_prefill([pkg], [A], k)
        _check(pkg, A, Y, k, where=f"{shape} k{k}")
    _status_ok()


def test_deterministic_and_reconstruction_consistent():
    """Two calls give identical bits, and a product with one-hot activation
    rows returns the bf16 reconstruction (rrq_reconstruct_ex) exactly."""
    rows, cols = 256, 1024
    W = workloads.generate(rows, cols, 9, "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], 128, 4, binding.GRID_SYM, binding.SCALE_F16)
    A = _acts(384, cols, seed=4)
    Y1 = binding.rrq_prefill([pkg], [A], 3)[0]
    Y2 = binding.rrq_prefill([pkg], [A], 3)[0]
    torch.cuda.synchronize()
    assert torch.equal(Y1.view(torch.int32), Y2.view(torch.int32))
    perm = torch.randperm(cols, generator=torch.Generator().manual_seed(1))
    E = torch.zeros((cols, cols), dtype=torch.bfloat16, device="cuda")
    E[torch.arange(cols), perm.cuda()] = 1.0
    for k in (1, 2, 3, 4):
        (Y,) = binding.rrq_prefill([pkg], [E], k)
        rec = binding.rrq_reconstruct_ex([pkg], k)[0][0]
        assert torch.equal(Y, rec.float()[:, perm.cuda()].T.contiguous()), f"k={k}"
    _status_ok()


@pytest.mark.parametrize("shape", [(129, 4096, 257), (256, 4096, 257), (300, 2048, 600), (129, 4096, 1500),
                                   (256, 2048, 2048)])
def test_repeated_runs_identical(shape):
    """The ring protocols leave no race: five runs of the same call give the
    same bits, and they match the oracle (ragged row and token tiles, the
    code tiles by TMA)."""
    rows, cols, tokens = shape
    W = workloads.generate(rows, cols, rows + cols, "t3", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], 128, 4, binding.GRID_ASYM, binding.SCALE_F32)
    A = _acts(tokens, cols, seed=rows)
    for k in (1, 4):
        outs = [binding.rrq_prefill([pkg], [A], k)[0] for _ in range(5)]
        torch.cuda.synchronize()
        for Y in outs[1:]:
            assert torch.equal(Y.view(torch.int32), outs[0].view(torch.int32)), f"{shape} k{k}: runs differ"
        _check(pkg, A, outs[0], k, where=f"{shape} k{k}")
    _status_ok()


def test_batch_across_launches():
    rng = np.random.default_rng(21)
    shapes = [(int(rng.integers(1, 300)), 128 * int(rng.integers(1, 12))) for _ in range(20)]
    mats = [workloads.generate(r, c, 1300 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    acts = [_acts(200, c, seed=i) for i, (r, c) in enumerate(shapes)]
    ys = binding.rrq_prefill(pkgs, acts, 2)
    for i, (p, A, Y) in enumerate(zip(pkgs, acts, ys)):
        _check(p, A, Y, 2, where=f"item {i}")
    _status_ok()


def test_qwen3_8b_layer_sampled():
    """A full-size Qwen3-8B-shaped layer (7 matrices, one call) at 2048
    tokens, every prefix: 48 sampled rows x 48 sampled tokens of every
    matrix against the oracle."""
    specs = workloads.config_matrices("qwen3_8b_layer")
    mats = [workloads.generate_spec(sp, "cuda") for sp in specs]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    tokens = 2048
    acts = [_acts(tokens, sp.cols, seed=60 + i) for i, sp in enumerate(specs)]
    for k in (1, 2, 3, 4):
        ys = binding.rrq_prefill(pkgs, acts, k)
        for i, (sp, p, A, Y) in enumerate(zip(specs, pkgs, acts, ys)):
            rng = np.random.default_rng(i * 10 + k)
            ridx = np.unique(np.concatenate([[0, sp.rows - 1], rng.integers(0, sp.rows, 46)]))
            tidx = np.unique(np.concatenate([[0, tokens - 1], rng.integers(0, tokens, 46)]))
            _check(p, A, Y, k, rows_idx=ridx, tok_idx=tidx, where=f"{sp.name} k{k}")
        del ys
    _status_ok()


@pytest.mark.parametrize("group", [32, 128])
@pytest.mark.parametrize("bits", [(1, 3), (3, 1), (4, 2, 1), (2, 4), (1, 1, 1, 1), (4, 4)],
                         ids=lambda b: "+".join(map(str, b)))
def test_widths(bits, group):
    """Packages with per-stage widths: every prefix against the oracle's
    prefill form (bf16 prefix weights) within the same bound, and one-hot
    rows returning the width reconstruction (rrq_reconstruct_ex) exactly."""
    rows, cols, tokens = 200, 8 * group, 600
    W = workloads.generate(rows, cols, 90 + sum(bits), "t3_rowout", "cuda")
    (pkg,) = binding.rrq_quantize_ex([W], group, len(bits), binding.GRID_ASYM, binding.SCALE_F32, bits=bits)
    A = _acts(tokens, cols, seed=len(bits) + group)
    torch.cuda.synchronize()
    codes = [c.cpu().numpy() for c in pkg.codes]
    scales = [x.cpu().numpy() for x in pkg.scales]
    zeros = [x.cpu().numpy() for x in pkg.zeros]
    Ab = bf16_bits(A)
    Af = np.abs((Ab.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
    perm = torch.randperm(cols, generator=torch.Generator().manual_seed(group))
    E = torch.zeros((cols, cols), dtype=torch.bfloat16, device="cuda")
    E[torch.arange(cols), perm.cuda()] = 1.0
    for k in range(1, len(bits) + 1):
        (Y,) = binding.rrq_prefill([pkg], [A], k)
        want = oracle.product_bits(codes, scales, zeros, rows, cols, group, k, bits, Ab, True)
        rec = oracle.reconstruct_bits(codes, scales, zeros, rows, cols, group, k, bits)
        recf = np.abs((rec.astype(np.uint32) << 16).view(np.float32).astype(np.float64))
        tol = (cols / 16 + 2) * 2.0 ** -23 * (Af @ recf.T) + 1e-30
        err = np.abs(Y.cpu().numpy().astype(np.float64) - want)
        assert not np.any(err > tol), f"{bits} g{group} k{k}: {int((err > tol).sum())} outputs beyond the bound"
        (Yh,) = binding.rrq_prefill([pkg], [E], k)
        rec_gpu = binding.rrq_reconstruct_ex([pkg], k)[0][0]
        assert torch.equal(Yh, rec_gpu.float()[:, perm.cuda()].T.contiguous()), f"{bits} g{group} k{k}: one-hot"
    _status_ok()


def test_errors():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    pkg = binding.rrq_quantize(W, 128, 2)
    A = _acts(4, 256, seed=1)
    with pytest.raises(ValueError):
        binding.rrq_prefill([pkg], [A], 3)  # k beyond the package
    Yover = A.view(torch.float32).reshape(-1)[:32].view(4, 8)  # Y over the activations
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_prefill([pkg], [A], 1, ys=[Yover])
    assert e.value.status == 1
    _status_ok()


def test_bounded_waits_report_timeout():
    """A wait limit of 0 makes every wait give up at once: the call reports
    RRQ_ERR_TIMEOUT through the status word, and the next call is exact."""
    W = workloads.generate(256, 1024, 2, "t3", "cuda")
    pkg = binding.rrq_quantize(W, 128, 4)
    A = _acts(300, 1024, seed=3)
    binding.rrq_set_wait_limit_us(0)
    try:
        binding.rrq_prefill([pkg], [A], 4)
        assert binding.rrq_get_device_status() == 5
    finally:
        binding.rrq_set_wait_limit_us(1000000)
    (Y,) = binding.rrq_prefill([pkg], [A], 4)
    _check(pkg, A, Y, 4, where="after timeout")
    _status_ok()


def test_guard_bands_untouched():
    """Outputs inside 4 KiB sentinel bands: a ragged row tile, a ragged token
    tile and a half stage, at k = 1 and 4 (one and four-CTA clusters)."""
    shapes = [(45, 288), (130, 4096 + 128)]
    mats = [workloads.generate(r, c, 700 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = [binding.rrq_quantize_ex([W], 32, 4, binding.GRID_ASYM, binding.SCALE_F32)[0] for W in mats]
    tokens = 1100
    acts = [_acts(tokens, c, seed=80 + i) for i, (r, c) in enumerate(shapes)]
    for k in (1, 4):
        bufs, ys, guard = guarded_outputs(shapes, tokens)
        binding.rrq_prefill(pkgs, acts, k, ys)
        assert bands_intact(bufs, guard), f"k {k}: a sentinel band changed"
        for i, (p, A, Y) in enumerate(zip(pkgs, acts, ys)):
            _check(p, A, Y, k, where=f"guarded item {i} k{k}")
