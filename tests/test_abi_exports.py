"""The C-ABI library loads and exports every function include/rrq.h declares;
argument checks that run before any CUDA call reject bad input (CPU only,
nothing is computed)."""
import ctypes
import os
import re

import pytest

from paper_2608_04048_gb300 import binding, build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "rrq.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rrq_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load_library()


def test_header_declares_the_boundary():
    names = declared_functions()
    assert "rrq_quantize" in names and "rrq_reconstruct" in names
    assert set(names) == set(binding.EXPORTS)


def test_binding_limits_match_the_header():
    defines = dict(re.findall(r"#define\s+(RRQ_[A-Z_0-9]+)\s+\(?([0-9]+)", open(HEADER).read()))
    assert int(defines["RRQ_MAX_STAGES"]) == binding.MAX_STAGES
    assert int(defines["RRQ_MAX_GEMV_BATCH"]) == binding.MAX_GEMV_BATCH
    assert int(defines["RRQ_MAX_GEMV_COLS"]) == binding.MAX_GEMV_COLS


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_size_helpers(lib):
    assert binding.rrq_codes_bytes(4096, 4096) == 4096 * 4096 // 4
    assert binding.rrq_meta_count(4096, 4096, 128) == 4096 * 4096 // 128
    assert binding.rrq_package_bytes(4096, 4096, 128, 4) == 4 * (4096 * 1024 + 8 * 4096 * 32)
    assert binding.rrq_meta_count(4, 100, 128) == 0
    assert binding.rrq_codes_bytes(0, 128) == 0
    assert binding.rrq_package_bytes(4, 128, 128, 5) == 0


def test_status_strings(lib):
    for code in range(6):
        assert lib.rrq_status_string(code).startswith(b"RRQ_")


def _call_quantize(lib, W, rows, cols, group, n_stages, codes, scales, zeros):
    arr = lambda xs: (ctypes.c_void_p * len(xs))(*xs)
    return lib.rrq_quantize(W, rows, cols, group, n_stages, arr(codes), arr(scales), arr(zeros), None)


def test_quantize_argument_checks_run_before_cuda(lib):
    base = 1 << 20
    ok = dict(W=base, rows=4, cols=256, group=128, n_stages=2,
              codes=[base + 0x10000, base + 0x20000], scales=[base + 0x30000, base + 0x40000],
              zeros=[base + 0x50000, base + 0x60000])

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        return _call_quantize(lib, a["W"], a["rows"], a["cols"], a["group"], a["n_stages"],
                              a["codes"], a["scales"], a["zeros"])

    assert call(W=None) == 1
    assert call(rows=0) == 1
    assert call(n_stages=0) == 1
    assert call(n_stages=5) == 1
    assert call(group=48) == 2
    assert call(group=512) == 2
    assert call(cols=192) == 1                      # cols % group != 0
    assert call(W=base + 8) == 3                    # bf16 input must be 16-byte aligned
    assert call(codes=[base + 0x10004, base + 0x20000]) == 3
    assert call(codes=[base + 0x10008, base + 0x20000]) == 3   # package arrays: 16-byte aligned
    assert call(scales=[base + 0x30002, base + 0x40000]) == 3
    assert call(codes=[base + 0x10000, base + 0x10040]) == 1   # overlapping outputs
    assert call(zeros=[base + 0x50000, base + 0x100]) == 1     # output overlaps W


def test_reconstruct_argument_checks_run_before_cuda(lib):
    base = 1 << 20
    arr = lambda xs: (ctypes.c_void_p * len(xs))(*xs)
    codes, scales, zeros = arr([base]), arr([base + 0x10000]), arr([base + 0x20000])
    assert lib.rrq_reconstruct(codes, scales, zeros, 4, 256, 128, 0, base + 0x40000, None) == 1
    assert lib.rrq_reconstruct(codes, scales, zeros, 4, 256, 100, 1, base + 0x40000, None) == 2
    assert lib.rrq_reconstruct(codes, scales, zeros, 4, 256, 128, 1, base + 0x40008, None) == 3
    assert lib.rrq_reconstruct(codes, scales, zeros, 4, 256, 128, 1, base + 0x80, None) == 1


def test_binding_refuses_cpu_tensors(lib):
    import torch
    with pytest.raises(TypeError):
        binding.rrq_quantize(torch.zeros(4, 128, dtype=torch.bfloat16))


def _fmt(group=128, n_stages=4, grid=1, scale_type=1):
    return binding.Format(group, n_stages, grid, scale_type)


def test_format_size_helpers(lib):
    n, g = 4096 * 4096, 128
    assert binding.rrq_scales_bytes(4096, 4096, g, binding.GRID_SYM, binding.SCALE_F16) == 2 * n // g
    assert binding.rrq_scales_bytes(4096, 4096, g, binding.GRID_SYM, binding.SCALE_F32) == 4 * n // g
    assert binding.rrq_scales_bytes(4096, 4096, g, binding.GRID_ASYM, binding.SCALE_F32) == 4 * n // g
    assert binding.rrq_scales_bytes(4096, 4096, g, binding.GRID_ASYM, binding.SCALE_F16) == 0
    # symmetric binary16 package: 2 bits + 16/128 bits per weight and stage
    assert binding.rrq_package_bytes_ex(4096, 4096, g, 4, binding.GRID_SYM, binding.SCALE_F16) == \
        4 * (n // 4 + 2 * n // g)
    assert binding.rrq_package_bytes_ex(4096, 4096, g, 4, binding.GRID_ASYM, binding.SCALE_F32) == \
        binding.rrq_package_bytes(4096, 4096, g, 4)
    assert binding.rrq_package_bytes_ex(4096, 4096, g, 5, binding.GRID_SYM, binding.SCALE_F16) == 0


def test_ex_argument_checks_run_before_cuda(lib):
    import torch
    base = 1 << 20
    no_device = 4 if not torch.cuda.is_available() else 1  # past the checks: CUDA error or not device memory

    def quantize(fmt, scales=(0x30000, 0x40000), zeros=(0, 0), W=base, count=1):
        d = binding.QuantizeDesc()
        d.W_bf16, d.rows, d.cols = W, 4, 256
        d.codes[0], d.codes[1] = base + 0x10000, base + 0x20000
        d.scales[0], d.scales[1] = base + scales[0], base + scales[1]
        d.zeros[0] = base + zeros[0] if zeros[0] else None
        d.zeros[1] = base + zeros[1] if zeros[1] else None
        items = (binding.QuantizeDesc * 1)(d)
        return lib.rrq_quantize_ex(items, count, ctypes.byref(fmt) if fmt is not None else None, None)

    assert quantize(None) == 1
    assert quantize(_fmt(n_stages=2, grid=2)) == 1
    assert quantize(_fmt(n_stages=2, scale_type=3)) == 1
    assert quantize(_fmt(n_stages=2, grid=0, scale_type=1)) == 2   # binary16 scales need the symmetric grid
    assert quantize(_fmt(group=48, n_stages=2)) == 2
    assert quantize(_fmt(n_stages=2), count=0) == 1
    assert quantize(_fmt(n_stages=2, grid=0, scale_type=0)) == 1   # asymmetric grid needs zeros
    assert quantize(_fmt(n_stages=2), scales=(0x30002, 0x40000)) == 3
    # 8 groups: binary16 scales span 16 bytes, binary32 scales 32 bytes
    assert quantize(_fmt(n_stages=2, scale_type=0), scales=(0x30000, 0x30010)) == 1
    assert quantize(_fmt(n_stages=2, scale_type=1), scales=(0x30000, 0x30010)) == no_device
    assert quantize(_fmt(n_stages=2, scale_type=1), scales=(0x30000, 0x3000F)) == 3

    r = binding.ReconstructDesc()
    r.codes[0], r.scales[0], r.rows, r.cols = base, base + 0x10000, 4, 256
    r.out_bf16[0] = base + 0x40000
    items = (binding.ReconstructDesc * 1)(r)
    assert lib.rrq_reconstruct_ex(items, 1, ctypes.byref(_fmt(n_stages=1)), 2, 0, None) == 1  # k > n_stages
    assert lib.rrq_reconstruct_ex(items, 1, ctypes.byref(_fmt(n_stages=1)), 1, 1, None) == no_device
    r.out_bf16[0] = base + 0x10004
    items = (binding.ReconstructDesc * 1)(r)
    assert lib.rrq_reconstruct_ex(items, 1, ctypes.byref(_fmt(n_stages=1)), 1, 0, None) == 3


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """Without the built library every entry point raises: there is no CPU
    fallback to take its place."""
    import torch
    monkeypatch.setattr(binding, "_LIB", None)
    monkeypatch.setattr(binding, "library_path", lambda: str(tmp_path / "librrq.so"))
    with pytest.raises(RuntimeError, match="missing"):
        binding.load_library()
    with pytest.raises((RuntimeError, TypeError)):
        binding.rrq_quantize(torch.zeros(4, 128, dtype=torch.bfloat16))
