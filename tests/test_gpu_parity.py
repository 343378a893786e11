"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle, bit
for bit, on seeded inputs: packed codes, scales and zeros must be identical
and the bf16 reconstruction at every prefix must match with 0 ULP."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_04048_gb300 import binding, build, workloads
from gpu_helpers import bf16_bits, check_full, gpu_package_host, assert_package_equal

pytestmark = pytest.mark.gpu

GROUPS = (32, 64, 128, 256)


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    binding.load_library()
    binding.rrq_set_debug_flags(0)
    binding.rrq_set_wait_limit_us(1_000_000)
    yield
    binding.rrq_set_debug_flags(0)


def test_single_4096_full():
    """4096x4096, N(0, 0.02^2), seed 0, group 128, four stages: whole
    package and all four prefixes."""
    W = workloads.generate(4096, 4096, 0, "normal", "cuda")
    check_full(W, 128, 4, where="single_4096")


@pytest.mark.parametrize("group", GROUPS)
@pytest.mark.parametrize("dist", ["normal", "t3", "t3_rowout", "t3_col0.01"])
def test_groups_and_distributions(group, dist):
    # 333 rows x (5 groups) -> a ragged last chunk and several chunks per warp
    W = workloads.generate(333, 5 * group, 17 + group, dist, "cuda")
    check_full(W, group, 4, where=f"{dist} g{group}")


@pytest.mark.parametrize("n_stages", [1, 2, 3])
@pytest.mark.parametrize("group", GROUPS)
def test_fewer_stages(n_stages, group):
    W = workloads.generate(64, 4 * group, 5, "t3_rowout", "cuda")
    check_full(W, group, n_stages, where=f"S={n_stages} g{group}")


@pytest.mark.parametrize("shape", [(1, 32), (1, 64), (1, 128), (1, 256), (3, 256), (31, 32),
                                   (1, 1024 + 32), (7, 2304), (2049, 128)])
def test_small_and_ragged_shapes(shape):
    rows, cols = shape
    for g in GROUPS:
        if cols % g:
            continue
        W = workloads.generate(rows, cols, rows * 7 + cols, "t3", "cuda")
        check_full(W, g, 4, where=f"{shape} g{g}")


def _edge_matrix(rows, cols, group, seed):
    """Every group is one of: Gaussian, constant, signed zeros, an exact 4-level
    grid with ties, a bf16-subnormal range, huge magnitudes, or a zero
    minimum with a -0 present."""
    rng = np.random.default_rng(seed)
    n_groups = rows * cols // group
    out = np.empty((n_groups, group), np.uint16)

    def bf16(x):
        u = np.asarray(x, np.float32).view(np.uint32)
        return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)

    for gi in range(n_groups):
        kind = gi % 8
        if kind == 0:
            out[gi] = bf16(rng.normal(0, 0.02, group))
        elif kind == 1:
            out[gi] = bf16(np.full(group, rng.normal(0, 1)))
        elif kind == 2:
            out[gi] = rng.choice(np.array([0x0000, 0x8000], np.uint16), group)
        elif kind == 3:
            a, d = int(rng.integers(-60, 60)), int(rng.integers(1, 60))
            q = rng.integers(0, 4, group) / 2.0  # half-steps: exact ties at .5
            q[0], q[-1] = 0, 3
            out[gi] = bf16((a + q * d) / 1024.0)
        elif kind == 4:
            out[gi] = rng.integers(0, 0x80, group).astype(np.uint16) | \
                (rng.integers(0, 2, group).astype(np.uint16) << 15)
        elif kind == 5:
            out[gi] = bf16(rng.normal(0, 1e30, group))
        elif kind == 6:
            v = bf16(np.abs(rng.normal(0, 0.02, group)))
            v[rng.integers(0, group)] = 0x8000
            v[rng.integers(0, group)] = 0x0000
            out[gi] = v
        else:
            out[gi] = bf16(rng.standard_t(3, group) * 0.02)
    W = torch.from_numpy(out.reshape(rows, cols).view(np.int16)).view(torch.bfloat16)
    return W.cuda()


@pytest.mark.parametrize("group", GROUPS)
def test_edge_case_groups(group):
    W = _edge_matrix(40, 8 * group, group, seed=group)
    check_full(W, group, 4, where=f"edge g{group}")


@pytest.mark.parametrize("group", GROUPS)
def test_forced_exact_path_matches(group):
    """The per-element IEEE-division path, forced for every group, gives the
    same bits as the oracle (and therefore as the default path)."""
    W = workloads.generate(96, 4 * group, 3, "t3_rowout", "cuda")
    binding.rrq_set_debug_flags(1)
    try:
        check_full(W, group, 4, where=f"forced-exact g{group}")
    finally:
        binding.rrq_set_debug_flags(0)
    W = _edge_matrix(16, 8 * group, group, seed=100 + group)
    binding.rrq_set_debug_flags(1)
    try:
        check_full(W, group, 4, where=f"forced-exact edge g{group}")
    finally:
        binding.rrq_set_debug_flags(0)


def test_guard_bands_untouched():
    """Outputs written only inside their extents: every output lives between
    two 4 KiB sentinel bands that must survive both kernels."""
    rows, cols, g, S = 77, 3 * 128, 128, 4
    n = rows * cols
    guard = 4096
    W = workloads.generate(rows, cols, 9, "t3_rowout", "cuda")

    def guarded(nbytes):
        buf = torch.full((nbytes + 2 * guard,), 0xA5, dtype=torch.uint8, device="cuda")
        return buf, buf[guard:guard + nbytes]

    bufs = []
    codes, scales, zeros = [], [], []
    for _ in range(S):
        b, c = guarded(n // 4); bufs.append(b); codes.append(c)
        b, s = guarded(4 * n // g); bufs.append(b); scales.append(s.view(torch.float32))
        b, z = guarded(4 * n // g); bufs.append(b); zeros.append(z.view(torch.float32))
    pkg = binding.Package(codes, scales, zeros, rows, cols, g, S)
    binding.rrq_quantize(W, g, S, out=pkg)
    ob, o = guarded(2 * n)
    binding.rrq_reconstruct(pkg, 4, out=o.view(torch.bfloat16).view(rows, cols))
    torch.cuda.synchronize()
    for b in bufs + [ob]:
        h = b.cpu().numpy()
        assert (h[:guard] == 0xA5).all() and (h[-guard:] == 0xA5).all()
    ref = oracle.quantize(bf16_bits(W), g, S)
    assert_package_equal(gpu_package_host(pkg), ref, S, "guarded")


def test_timeout_path_reports_and_recovers():
    """A wait limit of 0 makes every bounded wait give up at once: the kernel
    records RRQ_ERR_TIMEOUT, drains its own copies and returns; the device
    stays usable and the next call is exact again.  Both builds (the 2-D
    tile form and the 1-D ring form) and the one-prefix reconstruction of a
    whole number of 2048-weight chunks wait on barriers: the builds and that
    reconstruction up to k = 2 on bulk copies, from k = 3 on per-lane
    copies; the reconstruction of other sizes has no bounded waits."""
    W = workloads.generate(512, 1024, 21, "normal", "cuda")      # tile forms
    V = workloads.generate(3, 1024 + 32, 22, "normal", "cuda")   # 1-D forms (n % 64 != 0)
    binding.rrq_get_device_status()  # clear
    pkg = binding.rrq_quantize(W, 128, 4)
    pkv = binding.rrq_quantize(V, 32, 4)
    binding.rrq_set_wait_limit_us(0)
    try:
        binding.rrq_quantize(W, 128, 4)
        assert binding.rrq_get_device_status() == 5
        binding.rrq_quantize(V, 32, 4)
        assert binding.rrq_get_device_status() == 5
        binding.rrq_reconstruct(pkg, 4)
        assert binding.rrq_get_device_status() == 5
        binding.rrq_reconstruct(pkg, 2)
        assert binding.rrq_get_device_status() == 5
        binding.rrq_reconstruct(pkv, 4)  # cp.async copies complete in hardware
        assert binding.rrq_get_device_status() == 0
    finally:
        binding.rrq_set_wait_limit_us(1_000_000)
    assert binding.rrq_get_device_status() == 0
    check_full(W, 128, 4, where="after timeout")
    check_full(V, 32, 4, where="after timeout, 1-D forms")


def test_bad_pointers_rejected_on_device():
    W = workloads.generate(8, 256, 1, "normal", "cuda")
    host = torch.zeros(8 * 256 // 4, dtype=torch.uint8)
    pkg = binding.Package.empty(8, 256, 128, 4)
    pkg.codes[1] = host
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize(W, 128, 4, out=pkg)
    assert e.value.status == 1


def test_nonzero_current_stream():
    """Launches follow the caller's stream."""
    W = workloads.generate(1024, 1024, 2, "t3", "cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        pkg = binding.rrq_quantize(W, 128, 4)
        out = binding.rrq_reconstruct(pkg, 4)
    s.synchronize()
    ref = oracle.quantize(bf16_bits(W), 128, 4)
    assert_package_equal(gpu_package_host(pkg), ref, 4, "stream")
    assert np.array_equal(bf16_bits(out), oracle.reconstruct(*ref, 1024, 1024, 128, 4))


def test_batch_matches_oracle_across_launches():
    """rrq_quantize_batch / rrq_reconstruct_batch over 70 matrices of mixed
    shapes (two launches of the 64-matrix batch kernel, chunks of different
    matrices interleaved across warps): every package and reconstruction
    equals the oracle's."""
    rng = np.random.default_rng(0)
    shapes = [(int(rng.integers(1, 40)), 128 * int(rng.integers(1, 12))) for _ in range(70)]
    mats = [workloads.generate(r, c, 100 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    outs = {k: binding.rrq_reconstruct_batch(pkgs, k) for k in (1, 2, 3, 4)}
    torch.cuda.synchronize()
    for i, (W, pkg) in enumerate(zip(mats, pkgs)):
        ref = oracle.quantize(bf16_bits(W), 128, 4)
        assert_package_equal(gpu_package_host(pkg), ref, 4, f"batch item {i}")
        for k in (1, 2, 3, 4):
            want = oracle.reconstruct(*ref, W.shape[0], W.shape[1], 128, k)
            assert np.array_equal(bf16_bits(outs[k][i]), want), f"batch item {i} k={k}"


def test_batch_rejects_overlapping_outputs():
    mats = [workloads.generate(8, 256, i, "normal", "cuda") for i in range(2)]
    pkgs = [binding.Package.empty(8, 256, 128, 4) for _ in range(2)]
    pkgs[1].codes[0] = pkgs[0].codes[0]  # two matrices writing the same codes
    with pytest.raises(binding.RRQError) as e:
        binding.rrq_quantize_batch(mats, pkgs, 128, 4)
    assert e.value.status == 1


@pytest.mark.parametrize("group", GROUPS)
def test_batch_group_sizes(group):
    mats = [workloads.generate(17 + i, group * (1 + i), 7 * i + group, "t3", "cuda") for i in range(5)]
    pkgs = binding.rrq_quantize_batch(mats, group=group, n_stages=3)
    outs = binding.rrq_reconstruct_batch(pkgs, 3)
    torch.cuda.synchronize()
    for W, pkg, out in zip(mats, pkgs, outs):
        ref = oracle.quantize(bf16_bits(W), group, 3)
        assert_package_equal(gpu_package_host(pkg), ref, 3, f"batch g{group}")
        assert np.array_equal(bf16_bits(out), oracle.reconstruct(*ref, W.shape[0], W.shape[1], group, 3))


@pytest.mark.parametrize("group", GROUPS)
def test_prefixes_single_matches_oracle(group):
    """rrq_reconstruct_prefixes: one pass writes every prefix, each equal to
    the oracle's reconstruction with that many stages."""
    W = _edge_matrix(24, 8 * group, group, seed=7 + group)
    pkg = binding.rrq_quantize(W, group, 4)
    for k in (1, 2, 3, 4):
        outs = binding.rrq_reconstruct_prefixes(pkg, k)
        torch.cuda.synchronize()
        ref = oracle.quantize(bf16_bits(W), group, 4)
        for j, o in enumerate(outs):
            want = oracle.reconstruct(*ref, W.shape[0], W.shape[1], group, j + 1)
            assert np.array_equal(bf16_bits(o), want), f"g{group} k={k} prefix {j + 1}"


def test_prefixes_batch_matches_oracle():
    rng = np.random.default_rng(3)
    shapes = [(int(rng.integers(1, 30)), 128 * int(rng.integers(1, 10))) for _ in range(67)]
    mats = [workloads.generate(r, c, 300 + i, "t3_rowout", "cuda") for i, (r, c) in enumerate(shapes)]
    pkgs = binding.rrq_quantize_batch(mats, group=128, n_stages=4)
    outs = binding.rrq_reconstruct_prefixes_batch(pkgs, 4)
    torch.cuda.synchronize()
    for i, W in enumerate(mats):
        ref = oracle.quantize(bf16_bits(W), 128, 4)
        for j in range(4):
            want = oracle.reconstruct(*ref, W.shape[0], W.shape[1], 128, j + 1)
            assert np.array_equal(bf16_bits(outs[i][j]), want), f"item {i} prefix {j + 1}"
