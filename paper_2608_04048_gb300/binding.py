"""Thin ctypes binding of the RRQ C ABI (include/rrq.h).

Argument marshalling only: every step of quantization and reconstruction runs
in the CUDA kernels of librrq.so.  PyTorch supplies device memory and the
current CUDA stream.  There is no CPU fallback: if the library is missing or
the tensors are not on a CUDA device, the call raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None

_STATUS = {0: "RRQ_OK", 1: "RRQ_ERR_INVALID_ARG", 2: "RRQ_ERR_UNSUPPORTED",
           3: "RRQ_ERR_MISALIGNED", 4: "RRQ_ERR_CUDA", 5: "RRQ_ERR_TIMEOUT"}

#: symbols declared in include/rrq.h
EXPORTS = ["rrq_quantize", "rrq_reconstruct", "rrq_quantize_batch", "rrq_reconstruct_batch",
           "rrq_reconstruct_prefixes", "rrq_reconstruct_prefixes_batch",
           "rrq_quantize_ex", "rrq_reconstruct_ex", "rrq_quantize_from_base", "rrq_gemv", "rrq_prefill",
           "rrq_stage_codes_bytes", "rrq_group_pmr", "rrq_quantize_prefixes", "rrq_scales_bytes", "rrq_package_bytes_ex",
           "rrq_codes_bytes", "rrq_meta_count",
           "rrq_package_bytes", "rrq_get_device_status", "rrq_set_wait_limit_us",
           "rrq_set_debug_flags", "rrq_status_string", "rrq_last_cuda_error", "rrq_check_buffer"]


MAX_STAGES = 4

#: rrq_grid / rrq_scale_type of include/rrq.h
GRID_ASYM, GRID_SYM = 0, 1
SCALE_F32, SCALE_F16 = 0, 1


class Format(ctypes.Structure):
    """rrq_format of include/rrq.h (bits: per-stage code widths, 0 = 2)"""
    _fields_ = [("group", ctypes.c_int), ("n_stages", ctypes.c_int), ("grid", ctypes.c_int),
                ("scale_type", ctypes.c_int), ("bits", ctypes.c_int * MAX_STAGES)]


class QuantizeDesc(ctypes.Structure):
    """rrq_quantize_desc of include/rrq.h"""
    _fields_ = [("W_bf16", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES)]


class GemvDesc(ctypes.Structure):
    """rrq_gemv_desc of include/rrq.h"""
    _fields_ = [("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("A_bf16", ctypes.c_void_p), ("Y", ctypes.c_void_p)]


MAX_GEMV_BATCH = 8
MAX_GEMV_COLS = 57344   # widest matrix rrq_gemv takes (RRQ_MAX_GEMV_COLS)


class PmrDesc(ctypes.Structure):
    """rrq_pmr_desc of include/rrq.h"""
    _fields_ = [("W_bf16", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("pmr", ctypes.c_void_p), ("stats", ctypes.c_void_p)]


class QuantizePrefixesDesc(ctypes.Structure):
    """rrq_quantize_prefixes_desc of include/rrq.h"""
    _fields_ = [("W_bf16", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES), ("out_bf16", ctypes.c_void_p * MAX_STAGES)]


class ReconstructDesc(ctypes.Structure):
    """rrq_reconstruct_desc of include/rrq.h"""
    _fields_ = [("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("out_bf16", ctypes.c_void_p * MAX_STAGES)]


class QuantizeItem(ctypes.Structure):
    """rrq_quantize_item of include/rrq.h"""
    _fields_ = [("W_bf16", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES)]


class ReconstructItem(ctypes.Structure):
    """rrq_reconstruct_item of include/rrq.h"""
    _fields_ = [("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("out_bf16", ctypes.c_void_p)]


class PrefixesItem(ctypes.Structure):
    """rrq_prefixes_item of include/rrq.h"""
    _fields_ = [("codes", ctypes.c_void_p * MAX_STAGES), ("scales", ctypes.c_void_p * MAX_STAGES),
                ("zeros", ctypes.c_void_p * MAX_STAGES), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("out_bf16", ctypes.c_void_p * MAX_STAGES)]


class RRQError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        msg = _STATUS.get(status, f"status {status}")
        if status == 4 and _LIB is not None:
            msg += f" (cudaError {_LIB.rrq_last_cuda_error()})"
        super().__init__(f"{what}: {msg}" if what else msg)


def library_path() -> str:
    return os.path.join(_HERE, "_build", "librrq.so")


def load_library():
    """Load librrq.so (built in-tree by paper_2608_04048_gb300.build)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with "
                           "`python -m paper_2608_04048_gb300.build` (or __graft_entry__.build())")
    lib = ctypes.CDLL(path)
    vp, i64, i32, u32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_uint32
    ptr_array = ctypes.POINTER(ctypes.c_void_p)
    lib.rrq_quantize.argtypes = [vp, i64, i64, i32, i32, ptr_array, ptr_array, ptr_array, vp]
    lib.rrq_quantize.restype = i32
    lib.rrq_reconstruct.argtypes = [ptr_array, ptr_array, ptr_array, i64, i64, i32, i32, vp, vp]
    lib.rrq_reconstruct.restype = i32
    lib.rrq_quantize_batch.argtypes = [ctypes.POINTER(QuantizeItem), i32, i32, i32, vp]
    lib.rrq_quantize_batch.restype = i32
    lib.rrq_reconstruct_batch.argtypes = [ctypes.POINTER(ReconstructItem), i32, i32, i32, vp]
    lib.rrq_reconstruct_batch.restype = i32
    lib.rrq_reconstruct_prefixes.argtypes = [ptr_array, ptr_array, ptr_array, i64, i64, i32, i32,
                                             ptr_array, vp]
    lib.rrq_reconstruct_prefixes.restype = i32
    lib.rrq_reconstruct_prefixes_batch.argtypes = [ctypes.POINTER(PrefixesItem), i32, i32, i32, vp]
    lib.rrq_reconstruct_prefixes_batch.restype = i32
    fmt_p = ctypes.POINTER(Format)
    lib.rrq_quantize_ex.argtypes = [ctypes.POINTER(QuantizeDesc), i32, fmt_p, vp]
    lib.rrq_quantize_ex.restype = i32
    lib.rrq_quantize_prefixes.argtypes = [ctypes.POINTER(QuantizePrefixesDesc), i32, fmt_p, vp]
    lib.rrq_quantize_prefixes.restype = i32
    lib.rrq_quantize_from_base.argtypes = [ctypes.POINTER(QuantizeDesc), i32, fmt_p, vp]
    lib.rrq_quantize_from_base.restype = i32
    lib.rrq_gemv.argtypes = [ctypes.POINTER(GemvDesc), i32, fmt_p, i32, i32, vp]
    lib.rrq_gemv.restype = i32
    lib.rrq_prefill.argtypes = [ctypes.POINTER(GemvDesc), i32, fmt_p, i32, ctypes.c_int64, vp]
    lib.rrq_prefill.restype = i32
    lib.rrq_reconstruct_ex.argtypes = [ctypes.POINTER(ReconstructDesc), i32, fmt_p, i32, i32, vp]
    lib.rrq_reconstruct_ex.restype = i32
    lib.rrq_group_pmr.argtypes = [ctypes.POINTER(PmrDesc), i32, i32, vp]
    lib.rrq_group_pmr.restype = i32
    lib.rrq_stage_codes_bytes.argtypes = [i64, i64, i32]
    lib.rrq_stage_codes_bytes.restype = ctypes.c_size_t
    lib.rrq_scales_bytes.argtypes = [i64, i64, fmt_p]
    lib.rrq_scales_bytes.restype = ctypes.c_size_t
    lib.rrq_package_bytes_ex.argtypes = [i64, i64, fmt_p]
    lib.rrq_package_bytes_ex.restype = ctypes.c_size_t
    lib.rrq_codes_bytes.argtypes = [i64, i64]
    lib.rrq_codes_bytes.restype = ctypes.c_size_t
    lib.rrq_meta_count.argtypes = [i64, i64, i32]
    lib.rrq_meta_count.restype = ctypes.c_size_t
    lib.rrq_package_bytes.argtypes = [i64, i64, i32, i32]
    lib.rrq_package_bytes.restype = ctypes.c_size_t
    lib.rrq_get_device_status.argtypes = [vp]
    lib.rrq_get_device_status.restype = i32
    lib.rrq_set_wait_limit_us.argtypes = [u32]
    lib.rrq_set_wait_limit_us.restype = None
    lib.rrq_set_debug_flags.argtypes = [u32]
    lib.rrq_set_debug_flags.restype = None
    lib.rrq_status_string.argtypes = [i32]
    lib.rrq_status_string.restype = ctypes.c_char_p
    lib.rrq_check_buffer.argtypes = [vp, ctypes.c_size_t]
    lib.rrq_check_buffer.restype = i32
    lib.rrq_last_cuda_error.argtypes = []
    lib.rrq_last_cuda_error.restype = i32
    _LIB = lib
    return lib


def _stream_handle(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _ptrs(tensors, n) -> ctypes.Array:
    return (ctypes.c_void_p * n)(*[t.data_ptr() for t in tensors[:n]])


@dataclass
class Package:
    """An RRQ package on the device: per stage a code array (uint8, n/4) and
    a scale array (n/group; float32, or float16 = IEEE binary16 for
    SCALE_F16), plus a zero array (float32, n/group) for the asymmetric grid
    (empty list for the symmetric grid)."""
    codes: list
    scales: list
    zeros: list
    rows: int
    cols: int
    group: int
    n_stages: int
    grid: int = GRID_ASYM
    scale_type: int = SCALE_F32
    bits: tuple = (2, 2, 2, 2)

    @classmethod
    def empty(cls, rows, cols, group=128, n_stages=4, device=None, grid=GRID_ASYM,
              scale_type=SCALE_F32, bits=None) -> "Package":
        device = device or torch.device("cuda", torch.cuda.current_device())
        n = rows * cols
        bits = tuple(bits) if bits else (2,) * n_stages
        sdt = torch.float16 if scale_type == SCALE_F16 else torch.float32
        zeros = [] if grid == GRID_SYM else \
            [torch.empty(n // group, dtype=torch.float32, device=device) for _ in range(n_stages)]
        return cls([torch.empty(n * bits[k] // 8, dtype=torch.uint8, device=device) for k in range(n_stages)],
                   [torch.empty(n // group, dtype=sdt, device=device) for _ in range(n_stages)],
                   zeros, rows, cols, group, n_stages, grid, scale_type, bits + (2,) * (4 - len(bits)))

    def format(self) -> Format:
        return Format(self.group, self.n_stages, self.grid, self.scale_type,
                      (ctypes.c_int * MAX_STAGES)(*self.bits[:MAX_STAGES]))

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in self.codes + self.scales + self.zeros)


def rrq_quantize(W: torch.Tensor, group: int = 128, n_stages: int = 4, out: Package | None = None,
                 stream=None) -> Package:
    """Build the RRQ package of a 2-D bf16 CUDA tensor (rows x cols, groups of
    `group` consecutive columns) through the C ABI."""
    lib = load_library()
    if W.dtype != torch.bfloat16 or W.dim() != 2 or not W.is_cuda:
        raise TypeError("W must be a 2-D bfloat16 CUDA tensor")
    if not W.is_contiguous():
        raise ValueError("W must be contiguous (row-major)")
    rows, cols = W.shape
    if out is None:
        out = Package.empty(rows, cols, group, n_stages, W.device)
    rc = lib.rrq_quantize(W.data_ptr(), rows, cols, group, n_stages, _ptrs(out.codes, n_stages),
                          _ptrs(out.scales, n_stages), _ptrs(out.zeros, n_stages), _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_quantize")
    return out


def rrq_reconstruct(pkg: Package, k: int, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """bf16 weights of the prefix with the first k stages (k=1..4 -> 2/4/6/8 bits)."""
    lib = load_library()
    if out is None:
        out = torch.empty((pkg.rows, pkg.cols), dtype=torch.bfloat16, device=pkg.codes[0].device)
    if out.dtype != torch.bfloat16 or not out.is_cuda or not out.is_contiguous():
        raise TypeError("out must be a contiguous bfloat16 CUDA tensor")
    if not 1 <= k <= pkg.n_stages:
        raise ValueError(f"k must be in 1..{pkg.n_stages}")
    rc = lib.rrq_reconstruct(_ptrs(pkg.codes, k), _ptrs(pkg.scales, k), _ptrs(pkg.zeros, k),
                             pkg.rows, pkg.cols, pkg.group, k, out.data_ptr(), _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_reconstruct")
    return out


def quantize_items(mats, pkgs) -> ctypes.Array:
    """Host array of rrq_quantize_item for matrices and their packages (build
    once and reuse: the pointers stay valid while the tensors live)."""
    items = (QuantizeItem * len(mats))()
    for it, W, pkg in zip(items, mats, pkgs):
        if W.dtype != torch.bfloat16 or W.dim() != 2 or not W.is_cuda or not W.is_contiguous():
            raise TypeError("every W must be a contiguous 2-D bfloat16 CUDA tensor")
        it.W_bf16 = W.data_ptr()
        it.rows, it.cols = W.shape
        for k in range(pkg.n_stages):
            it.codes[k] = pkg.codes[k].data_ptr()
            it.scales[k] = pkg.scales[k].data_ptr()
            it.zeros[k] = pkg.zeros[k].data_ptr()
    return items


def reconstruct_items(pkgs, outs) -> ctypes.Array:
    items = (ReconstructItem * len(pkgs))()
    for it, pkg, out in zip(items, pkgs, outs):
        if out.dtype != torch.bfloat16 or not out.is_cuda or not out.is_contiguous():
            raise TypeError("every out must be a contiguous bfloat16 CUDA tensor")
        for k in range(pkg.n_stages):
            it.codes[k] = pkg.codes[k].data_ptr()
            it.scales[k] = pkg.scales[k].data_ptr()
            it.zeros[k] = pkg.zeros[k].data_ptr()
        it.rows, it.cols = pkg.rows, pkg.cols
        it.out_bf16 = out.data_ptr()
    return items


def rrq_quantize_batch(mats, pkgs=None, group: int = 128, n_stages: int = 4, stream=None, items=None):
    """rrq_quantize for a list of matrices in one call (one launch per 64).
    Returns the packages; `items` may be a prebuilt quantize_items() array."""
    lib = load_library()
    if pkgs is None:
        pkgs = [Package.empty(W.shape[0], W.shape[1], group, n_stages, W.device) for W in mats]
    if items is None:
        items = quantize_items(mats, pkgs)
    rc = lib.rrq_quantize_batch(items, len(items), group, n_stages, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_quantize_batch")
    return pkgs


def rrq_reconstruct_batch(pkgs, k: int, outs=None, stream=None, items=None):
    """rrq_reconstruct at prefix k for a list of packages in one call."""
    lib = load_library()
    if outs is None:
        outs = [torch.empty((p.rows, p.cols), dtype=torch.bfloat16, device=p.codes[0].device) for p in pkgs]
    if items is None:
        items = reconstruct_items(pkgs, outs)
    group = pkgs[0].group
    if any(not 1 <= k <= p.n_stages for p in pkgs):
        raise ValueError("k exceeds the stages of a package")
    rc = lib.rrq_reconstruct_batch(items, len(items), group, k, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_reconstruct_batch")
    return outs


def _new_outs(pkg, k):
    return [torch.empty((pkg.rows, pkg.cols), dtype=torch.bfloat16, device=pkg.codes[0].device)
            for _ in range(k)]


def rrq_reconstruct_prefixes(pkg: Package, k: int, outs=None, stream=None):
    """bf16 weights of every prefix 1..k in one pass: outs[j] has j+1 stages."""
    lib = load_library()
    if not 1 <= k <= pkg.n_stages:
        raise ValueError(f"k must be in 1..{pkg.n_stages}")
    outs = outs if outs is not None else _new_outs(pkg, k)
    for o in outs:
        if o.dtype != torch.bfloat16 or not o.is_cuda or not o.is_contiguous():
            raise TypeError("outputs must be contiguous bfloat16 CUDA tensors")
    rc = lib.rrq_reconstruct_prefixes(_ptrs(pkg.codes, k), _ptrs(pkg.scales, k), _ptrs(pkg.zeros, k),
                                      pkg.rows, pkg.cols, pkg.group, k, _ptrs(outs, k),
                                      _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_reconstruct_prefixes")
    return outs


def prefixes_items(pkgs, outs, k) -> ctypes.Array:
    items = (PrefixesItem * len(pkgs))()
    for it, pkg, o in zip(items, pkgs, outs):
        for j in range(k):
            it.codes[j] = pkg.codes[j].data_ptr()
            it.scales[j] = pkg.scales[j].data_ptr()
            it.zeros[j] = pkg.zeros[j].data_ptr()
            if o[j].dtype != torch.bfloat16 or not o[j].is_cuda or not o[j].is_contiguous():
                raise TypeError("outputs must be contiguous bfloat16 CUDA tensors")
            it.out_bf16[j] = o[j].data_ptr()
        it.rows, it.cols = pkg.rows, pkg.cols
    return items


def rrq_reconstruct_prefixes_batch(pkgs, k: int, outs=None, stream=None, items=None):
    """rrq_reconstruct_prefixes for a list of packages: outs[i][j] is matrix
    i's prefix with j+1 stages."""
    lib = load_library()
    if any(not 1 <= k <= p.n_stages for p in pkgs):
        raise ValueError("k exceeds the stages of a package")
    if outs is None:
        outs = [_new_outs(p, k) for p in pkgs]
    if items is None:
        items = prefixes_items(pkgs, outs, k)
    rc = lib.rrq_reconstruct_prefixes_batch(items, len(items), pkgs[0].group, k, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_reconstruct_prefixes_batch")
    return outs


def quantize_descs(mats, pkgs) -> ctypes.Array:
    """Host array of rrq_quantize_desc for matrices and their packages."""
    items = (QuantizeDesc * len(mats))()
    for it, W, pkg in zip(items, mats, pkgs):
        if W.dtype != torch.bfloat16 or W.dim() != 2 or not W.is_cuda or not W.is_contiguous():
            raise TypeError("every W must be a contiguous 2-D bfloat16 CUDA tensor")
        it.W_bf16 = W.data_ptr()
        it.rows, it.cols = W.shape
        for k in range(pkg.n_stages):
            it.codes[k] = pkg.codes[k].data_ptr()
            it.scales[k] = pkg.scales[k].data_ptr()
            it.zeros[k] = pkg.zeros[k].data_ptr() if pkg.zeros else None
    return items


def rrq_quantize_ex(mats, group: int = 128, n_stages: int = 4, grid: int = GRID_SYM,
                    scale_type: int = SCALE_F16, pkgs=None, stream=None, items=None, bits=None):
    """Packages of a list of bf16 matrices in any supported format (one
    launch per 64 matrices).  Default: the symmetric grid with binary16
    scales.  bits: per-stage code widths (asymmetric grid), default 2."""
    lib = load_library()
    if pkgs is None:
        pkgs = [Package.empty(W.shape[0], W.shape[1], group, n_stages, W.device, grid, scale_type, bits)
                for W in mats]
    if items is None:
        items = quantize_descs(mats, pkgs)
    fmt = pkgs[0].format()
    fmt.group, fmt.n_stages, fmt.grid, fmt.scale_type = group, n_stages, grid, scale_type
    rc = lib.rrq_quantize_ex(items, len(items), ctypes.byref(fmt), _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_quantize_ex")
    return pkgs


def quantize_prefixes_descs(mats, pkgs, outs) -> ctypes.Array:
    """Host array of rrq_quantize_prefixes_desc; outs[i][j] is matrix i's
    prefix with j+1 stages (bf16, the matrix's shape)."""
    items = (QuantizePrefixesDesc * len(mats))()
    for it, W, pkg, o in zip(items, mats, pkgs, outs):
        if W.dtype != torch.bfloat16 or W.dim() != 2 or not W.is_cuda or not W.is_contiguous():
            raise TypeError("every W must be a contiguous 2-D bfloat16 CUDA tensor")
        it.W_bf16 = W.data_ptr()
        it.rows, it.cols = W.shape
        for k in range(pkg.n_stages):
            it.codes[k] = pkg.codes[k].data_ptr()
            it.scales[k] = pkg.scales[k].data_ptr()
            it.zeros[k] = pkg.zeros[k].data_ptr() if pkg.zeros else None
            if o[k].dtype != torch.bfloat16 or not o[k].is_cuda or not o[k].is_contiguous():
                raise TypeError("outputs must be contiguous bfloat16 CUDA tensors")
            it.out_bf16[k] = o[k].data_ptr()
    return items


def rrq_quantize_prefixes(mats, group: int = 128, n_stages: int = 4, grid: int = GRID_ASYM,
                          scale_type: int = SCALE_F32, pkgs=None, outs=None, stream=None, items=None):
    """Package of each matrix and its bf16 reconstruction after every stage,
    in one pass: returns (pkgs, outs) with outs[i][j] = prefix j+1."""
    lib = load_library()
    if pkgs is None:
        pkgs = [Package.empty(W.shape[0], W.shape[1], group, n_stages, W.device, grid, scale_type) for W in mats]
    if outs is None:
        outs = [_new_outs(p, n_stages) for p in pkgs]
    if items is None:
        items = quantize_prefixes_descs(mats, pkgs, outs)
    fmt = Format(group, n_stages, grid, scale_type)
    rc = lib.rrq_quantize_prefixes(items, len(items), ctypes.byref(fmt), _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_quantize_prefixes")
    return pkgs, outs


def rrq_quantize_from_base(mats, pkgs, stream=None, items=None):
    """Algorithm 1 with a base checkpoint: each package's stage 0 (codes[0],
    scales[0], zeros[0]) is given; stages 1.. are computed in place."""
    lib = load_library()
    if items is None:
        items = quantize_descs(mats, pkgs)
    fmt = pkgs[0].format()
    rc = lib.rrq_quantize_from_base(items, len(items), ctypes.byref(fmt), _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_quantize_from_base")
    return pkgs


def gemv_descs(pkgs, acts, ys, k) -> ctypes.Array:
    """Host array of rrq_gemv_desc: acts[i] bf16 [batch, cols], ys[i] float32
    [batch, rows]."""
    items = (GemvDesc * len(pkgs))()
    for it, pkg, A, Y in zip(items, pkgs, acts, ys):
        if A.dtype != torch.bfloat16 or A.dim() != 2 or not A.is_cuda or not A.is_contiguous():
            raise TypeError("activations must be contiguous 2-D bfloat16 CUDA tensors")
        if Y.dtype != torch.float32 or not Y.is_cuda or not Y.is_contiguous():
            raise TypeError("outputs must be contiguous float32 CUDA tensors")
        for j in range(k):
            it.codes[j] = pkg.codes[j].data_ptr()
            it.scales[j] = pkg.scales[j].data_ptr()
            it.zeros[j] = pkg.zeros[j].data_ptr() if pkg.zeros else None
        it.rows, it.cols = pkg.rows, pkg.cols
        it.A_bf16, it.Y = A.data_ptr(), Y.data_ptr()
    return items


def rrq_gemv(pkgs, acts, k: int, ys=None, stream=None, items=None):
    """Y_i = A_i W~_i^T for each package i at prefix k (Appendix C), A_i bf16
    [batch, cols] with 1 <= batch <= 8 and cols <= MAX_GEMV_COLS; returns
    float32 [batch, rows] each."""
    lib = load_library()
    batch = acts[0].shape[0]
    if any(not 1 <= k <= p.n_stages for p in pkgs):
        raise ValueError("k exceeds the stages of a package")
    if any(A.shape[0] != batch for A in acts):
        raise ValueError("every activation matrix must have the same batch")
    if ys is None:
        ys = [torch.empty((batch, p.rows), dtype=torch.float32, device=p.codes[0].device) for p in pkgs]
    if items is None:
        items = gemv_descs(pkgs, acts, ys, k)
    fmt = pkgs[0].format()
    rc = lib.rrq_gemv(items, len(items), ctypes.byref(fmt), k, batch, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_gemv")
    return ys


def rrq_prefill(pkgs, acts, k: int, ys=None, stream=None, items=None):
    """Y_i = A_i bf16(W~_i)^T for each package i at prefix k on the tensor
    cores (Appendix C's product for many activation rows), A_i bf16 [tokens,
    cols]; returns float32 [tokens, rows] each."""
    lib = load_library()
    tokens = acts[0].shape[0]
    if any(not 1 <= k <= p.n_stages for p in pkgs):
        raise ValueError("k exceeds the stages of a package")
    if any(A.shape[0] != tokens for A in acts):
        raise ValueError("every activation matrix must have the same number of tokens")
    if ys is None:
        ys = [torch.empty((tokens, p.rows), dtype=torch.float32, device=p.codes[0].device) for p in pkgs]
    if items is None:
        items = gemv_descs(pkgs, acts, ys, k)
    fmt = pkgs[0].format()
    rc = lib.rrq_prefill(items, len(items), ctypes.byref(fmt), k, tokens, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_prefill")
    return ys


def reconstruct_descs(pkgs, outs, k) -> ctypes.Array:
    """Host array of rrq_reconstruct_desc; outs[i] is a list of 1 or k outputs."""
    items = (ReconstructDesc * len(pkgs))()
    for it, pkg, o in zip(items, pkgs, outs):
        for j in range(k):
            it.codes[j] = pkg.codes[j].data_ptr()
            it.scales[j] = pkg.scales[j].data_ptr()
            it.zeros[j] = pkg.zeros[j].data_ptr() if pkg.zeros else None
        for j, t in enumerate(o):
            if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
                raise TypeError("outputs must be contiguous bfloat16 CUDA tensors")
            it.out_bf16[j] = t.data_ptr()
        it.rows, it.cols = pkg.rows, pkg.cols
    return items


def rrq_reconstruct_ex(pkgs, k: int, all_prefixes: bool = False, outs=None, stream=None, items=None):
    """Prefix reconstruction of packages of one format: outs[i] = [prefix k]
    or, with all_prefixes, [prefix 1, ..., prefix k]."""
    lib = load_library()
    if any(not 1 <= k <= p.n_stages for p in pkgs):
        raise ValueError("k exceeds the stages of a package")
    if outs is None:
        outs = [_new_outs(p, k if all_prefixes else 1) for p in pkgs]
    if items is None:
        items = reconstruct_descs(pkgs, outs, k)
    fmt = pkgs[0].format()
    rc = lib.rrq_reconstruct_ex(items, len(items), ctypes.byref(fmt), k, int(all_prefixes),
                                _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_reconstruct_ex")
    return outs


def rrq_group_pmr(mats, group: int = 128, stream=None):
    """Per-group peak-to-mean ratios (float32 [rows*cols/group]) and per-matrix
    [max, mean] (float32 [2]) of a list of bf16 matrices."""
    lib = load_library()
    items = (PmrDesc * len(mats))()
    pmrs, stats = [], []
    for it, W in zip(items, mats):
        if W.dtype != torch.bfloat16 or W.dim() != 2 or not W.is_cuda or not W.is_contiguous():
            raise TypeError("every W must be a contiguous 2-D bfloat16 CUDA tensor")
        pm = torch.empty(W.numel() // group, dtype=torch.float32, device=W.device)
        st = torch.empty(4, dtype=torch.float32, device=W.device)
        it.W_bf16, (it.rows, it.cols), it.pmr, it.stats = W.data_ptr(), W.shape, pm.data_ptr(), st.data_ptr()
        pmrs.append(pm)
        stats.append(st[:2])
    rc = lib.rrq_group_pmr(items, len(items), group, _stream_handle(stream))
    if rc != 0:
        raise RRQError(rc, "rrq_group_pmr")
    return pmrs, stats


def rrq_stage_codes_bytes(rows: int, cols: int, bits: int) -> int:
    return int(load_library().rrq_stage_codes_bytes(rows, cols, bits))


def rrq_scales_bytes(rows: int, cols: int, group: int, grid: int, scale_type: int,
                     n_stages: int = 4) -> int:
    return int(load_library().rrq_scales_bytes(rows, cols,
                                               ctypes.byref(Format(group, n_stages, grid, scale_type))))


def rrq_package_bytes_ex(rows: int, cols: int, group: int, n_stages: int, grid: int,
                         scale_type: int) -> int:
    return int(load_library().rrq_package_bytes_ex(
        rows, cols, ctypes.byref(Format(group, n_stages, grid, scale_type))))


def rrq_codes_bytes(rows: int, cols: int) -> int:
    return int(load_library().rrq_codes_bytes(rows, cols))


def rrq_meta_count(rows: int, cols: int, group: int) -> int:
    return int(load_library().rrq_meta_count(rows, cols, group))


def rrq_package_bytes(rows: int, cols: int, group: int, n_stages: int) -> int:
    return int(load_library().rrq_package_bytes(rows, cols, group, n_stages))


def rrq_get_device_status(stream=None) -> int:
    """Synchronizes the stream; returns 0 (RRQ_OK) or a status code."""
    return int(load_library().rrq_get_device_status(_stream_handle(stream)))


def rrq_check_buffer(ptr: int, nbytes: int) -> int:
    """Status of the library's device-buffer check for [ptr, ptr + nbytes)
    (0 = device memory of the current device; launches nothing)."""
    return int(load_library().rrq_check_buffer(ptr, nbytes))


def rrq_set_wait_limit_us(us: int) -> None:
    load_library().rrq_set_wait_limit_us(us)


def rrq_set_debug_flags(flags: int) -> None:
    load_library().rrq_set_debug_flags(flags)
