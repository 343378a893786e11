"""RRQ CPU oracle: TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg (and its ``--impl reference`` arm) may import this package.  The product
path -- the CUDA library under ``paper_2608_04048_gb300`` -- never imports it,
and the two share no code.

This module compiles ``rrq_oracle.c`` with gcc (``-O2 -ffp-contract=off``, no
fast-math) and exposes it to numpy through ctypes.  The arithmetic itself lives
in the C file, which cites the paper's equations step by step (Section 3.1
Eq. 1-3, Section 3.2 Eq. 4-8, Algorithm 1), for the asymmetric min/max grid
and for the symmetric grid with binary32 or binary16 scales.

Every function here is pinned by ``tests/test_oracle_pins.py`` (hand-worked
groups, brute-force nearest level, invariants) and
``tests/test_oracle_mutants.py`` (planted mistakes fail the pins).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rrq_oracle.c")
_HDR = os.path.join(_HERE, "rrq_oracle.h")
_BUILD_DIR = os.path.join(_HERE, "_build")
LIB_PATH = os.path.join(_BUILD_DIR, "liboracle_rrq.so")

CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def compile_oracle(src: str = _SRC, out: str = LIB_PATH, extra_flags=()) -> str:
    """Compile an oracle source file into a shared library (atomic replace)."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=os.path.dirname(out))
    os.close(fd)
    cmd = ["gcc", *CFLAGS, *extra_flags, "-I", _HERE, "-o", tmp, src, "-lm"]
    try:
        subprocess.run(cmd, check=True, capture_output=True, text=True)
    except subprocess.CalledProcessError as e:  # pragma: no cover - build failure
        os.unlink(tmp)
        raise RuntimeError(f"oracle build failed: {' '.join(cmd)}\n{e.stderr}") from e
    os.replace(tmp, out)
    return out


def build() -> str:
    """Build the oracle library if it is missing or older than its sources."""
    if os.path.exists(LIB_PATH):
        t = os.path.getmtime(LIB_PATH)
        if t >= os.path.getmtime(_SRC) and t >= os.path.getmtime(_HDR):
            return LIB_PATH
    return compile_oracle()


_u8p = ctypes.POINTER(ctypes.c_uint8)
_f32p = ctypes.POINTER(ctypes.c_float)
_u16p = ctypes.POINTER(ctypes.c_uint16)


class Oracle:
    """ctypes view of one compiled oracle library (the committed one, or a
    test's mutated copy)."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        lib.rrq_oracle_quantize_group.argtypes = [
            _f32p, ctypes.c_int, ctypes.c_int, _u8p, _f32p, _f32p, _f32p]
        lib.rrq_oracle_quantize_group.restype = ctypes.c_int
        lib.rrq_oracle_quantize.argtypes = [
            _u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int,
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p)]
        lib.rrq_oracle_quantize.restype = ctypes.c_int
        lib.rrq_oracle_reconstruct.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p),
            ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _u16p]
        lib.rrq_oracle_reconstruct.restype = ctypes.c_int
        lib.rrq_oracle_f32_to_bf16.argtypes = [ctypes.c_float]
        lib.rrq_oracle_f32_to_bf16.restype = ctypes.c_uint16
        lib.rrq_oracle_quantize_group_sym.argtypes = [
            _f32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _u8p, _f32p, _f32p]
        lib.rrq_oracle_quantize_group_sym.restype = ctypes.c_int
        lib.rrq_oracle_quantize_sym.argtypes = [
            _u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.POINTER(_u8p), ctypes.POINTER(ctypes.c_void_p)]
        lib.rrq_oracle_quantize_sym.restype = ctypes.c_int
        lib.rrq_oracle_reconstruct_sym.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(ctypes.c_void_p), ctypes.c_int64, ctypes.c_int64,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, _u16p]
        lib.rrq_oracle_reconstruct_sym.restype = ctypes.c_int
        lib.rrq_oracle_quantize_from_base.argtypes = [
            _u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_int, ctypes.POINTER(_u8p), ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(_f32p)]
        lib.rrq_oracle_quantize_from_base.restype = ctypes.c_int
        lib.rrq_oracle_gemv.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(_f32p),
            ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            _u16p, ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
        lib.rrq_oracle_gemv.restype = ctypes.c_int
        lib.rrq_oracle_prefill.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(_f32p),
            ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            _u16p, ctypes.c_int64, ctypes.POINTER(ctypes.c_double)]
        lib.rrq_oracle_prefill.restype = ctypes.c_int
        _i32p = ctypes.POINTER(ctypes.c_int)
        lib.rrq_oracle_quantize_group_bits.argtypes = [
            _f32p, ctypes.c_int, ctypes.c_int, _i32p, _u8p, _f32p, _f32p, _f32p]
        lib.rrq_oracle_quantize_group_bits.restype = ctypes.c_int
        lib.rrq_oracle_quantize_bits.argtypes = [
            _u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _i32p,
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p)]
        lib.rrq_oracle_quantize_bits.restype = ctypes.c_int
        lib.rrq_oracle_reconstruct_bits.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p),
            ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _i32p, _u16p]
        lib.rrq_oracle_reconstruct_bits.restype = ctypes.c_int
        lib.rrq_oracle_product_bits.argtypes = [
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p), ctypes.c_int64, ctypes.c_int64,
            ctypes.c_int, ctypes.c_int, _i32p, _u16p, ctypes.c_int64, ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
        lib.rrq_oracle_product_bits.restype = ctypes.c_int
        lib.rrq_oracle_quantize_from_base_bits.argtypes = [
            _u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _i32p,
            ctypes.POINTER(_u8p), ctypes.POINTER(_f32p), ctypes.POINTER(_f32p)]
        lib.rrq_oracle_quantize_from_base_bits.restype = ctypes.c_int
        lib.rrq_oracle_group_pmr.argtypes = [_u16p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                                             ctypes.POINTER(ctypes.c_double)]
        lib.rrq_oracle_group_pmr.restype = ctypes.c_int
        lib.rrq_oracle_f32_to_f16.argtypes = [ctypes.c_float]
        lib.rrq_oracle_f32_to_f16.restype = ctypes.c_uint16
        lib.rrq_oracle_f16_to_f32.argtypes = [ctypes.c_uint16]
        lib.rrq_oracle_f16_to_f32.restype = ctypes.c_float
        self.lib = lib

    # -- one group, float input, unpacked codes --------------------------------
    def quantize_group(self, x, n_stages: int = 4):
        """Returns (Q[n_stages, g] uint8, scale[n_stages] f32, zero[n_stages] f32,
        resid[n_stages, g] f32) for one group of float32 values."""
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
        g = x.size
        Q = np.zeros((n_stages, g), np.uint8)
        s = np.zeros(n_stages, np.float32)
        z = np.zeros(n_stages, np.float32)
        r = np.zeros((n_stages, g), np.float32)
        rc = self.lib.rrq_oracle_quantize_group(
            x.ctypes.data_as(_f32p), g, n_stages, Q.ctypes.data_as(_u8p),
            s.ctypes.data_as(_f32p), z.ctypes.data_as(_f32p), r.ctypes.data_as(_f32p))
        if rc != 0:
            raise ValueError("oracle rejected the group")
        return Q, s, z, r

    # -- a bf16 matrix, packed package -----------------------------------------
    def quantize(self, W_bits, group: int = 128, n_stages: int = 4):
        """W_bits: uint16 array [rows, cols] of bf16 bit patterns.
        Returns (codes, scales, zeros): lists of n_stages numpy arrays."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        n = rows * cols
        codes = [np.zeros((n + 3) // 4, np.uint8) for _ in range(n_stages)]
        scales = [np.zeros(n // group, np.float32) for _ in range(n_stages)]
        zeros = [np.zeros(n // group, np.float32) for _ in range(n_stages)]
        cp = (_u8p * n_stages)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * n_stages)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * n_stages)(*[a.ctypes.data_as(_f32p) for a in zeros])
        rc = self.lib.rrq_oracle_quantize(W_bits.ctypes.data_as(_u16p), rows, cols,
                                          group, n_stages, cp, sp, zp)
        if rc != 0:
            raise ValueError("oracle rejected the matrix")
        return codes, scales, zeros

    def reconstruct(self, codes, scales, zeros, rows: int, cols: int, group: int, k: int):
        """bf16 bit patterns [rows, cols] of the prefix-k reconstruction."""
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=np.float32) for a in scales[:k]]
        zeros = [np.ascontiguousarray(a, dtype=np.float32) for a in zeros[:k]]
        out = np.zeros((rows, cols), np.uint16)
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in zeros])
        rc = self.lib.rrq_oracle_reconstruct(cp, sp, zp, rows, cols, group, k,
                                             out.ctypes.data_as(_u16p))
        if rc != 0:
            raise ValueError("oracle rejected the reconstruction")
        return out

    def f32_to_bf16(self, f: float) -> int:
        return int(self.lib.rrq_oracle_f32_to_bf16(ctypes.c_float(f)))

    def f32_to_f16(self, f: float) -> int:
        return int(self.lib.rrq_oracle_f32_to_f16(ctypes.c_float(f)))

    def f16_to_f32(self, h: int) -> float:
        return float(self.lib.rrq_oracle_f16_to_f32(ctypes.c_uint16(h)))

    # -- symmetric grid ----------------------------------------------------------
    def quantize_group_sym(self, x, n_stages: int = 4, scale_f16: bool = False):
        """Returns (Q[n_stages, g] uint8, scale[n_stages] f32 (the value used),
        resid[n_stages, g] f32) for one group under the symmetric grid."""
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
        g = x.size
        Q = np.zeros((n_stages, g), np.uint8)
        s = np.zeros(n_stages, np.float32)
        r = np.zeros((n_stages, g), np.float32)
        rc = self.lib.rrq_oracle_quantize_group_sym(
            x.ctypes.data_as(_f32p), g, n_stages, int(scale_f16), Q.ctypes.data_as(_u8p),
            s.ctypes.data_as(_f32p), r.ctypes.data_as(_f32p))
        if rc != 0:
            raise ValueError("oracle rejected the group")
        return Q, s, r

    def quantize_sym(self, W_bits, group: int = 128, n_stages: int = 4, scale_f16: bool = True):
        """Symmetric package of a bf16 matrix: (codes, scales) with scales
        float32 arrays, or uint16 binary16 bit patterns when scale_f16."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        n = rows * cols
        sdt = np.uint16 if scale_f16 else np.float32
        codes = [np.zeros((n + 3) // 4, np.uint8) for _ in range(n_stages)]
        scales = [np.zeros(n // group, sdt) for _ in range(n_stages)]
        cp = (_u8p * n_stages)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (ctypes.c_void_p * n_stages)(*[a.ctypes.data for a in scales])
        rc = self.lib.rrq_oracle_quantize_sym(W_bits.ctypes.data_as(_u16p), rows, cols, group,
                                              n_stages, int(scale_f16), cp, sp)
        if rc != 0:
            raise ValueError("oracle rejected the matrix")
        return codes, scales

    def quantize_from_base(self, W_bits, base, group: int = 128, n_stages: int = 4,
                           sym: bool = False, scale_f16: bool = False):
        """Algorithm 1 with a base checkpoint.  base = (codes0, scales0, zeros0)
        (zeros0 None for the symmetric grid).  Returns the whole package
        (codes, scales, zeros), stage 0 being the given base; zeros is None for
        the symmetric grid."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        n = rows * cols
        sdt = np.uint16 if scale_f16 else np.float32
        codes = [np.ascontiguousarray(base[0], dtype=np.uint8).copy()] + \
            [np.zeros((n + 3) // 4, np.uint8) for _ in range(n_stages - 1)]
        scales = [np.ascontiguousarray(base[1], dtype=sdt).copy()] + \
            [np.zeros(n // group, sdt) for _ in range(n_stages - 1)]
        cp = (_u8p * n_stages)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (ctypes.c_void_p * n_stages)(*[a.ctypes.data for a in scales])
        zeros = None
        zp = None
        if not sym:
            zeros = [np.ascontiguousarray(base[2], dtype=np.float32).copy()] + \
                [np.zeros(n // group, np.float32) for _ in range(n_stages - 1)]
            zp = (_f32p * n_stages)(*[a.ctypes.data_as(_f32p) for a in zeros])
        rc = self.lib.rrq_oracle_quantize_from_base(W_bits.ctypes.data_as(_u16p), rows, cols, group,
                                                    n_stages, int(sym), int(scale_f16), cp, sp, zp)
        if rc != 0:
            raise ValueError("oracle rejected the base-checkpoint build")
        return codes, scales, zeros

    def gemv(self, codes, scales, zeros, rows: int, cols: int, group: int, k: int, A_bits,
             sym: bool = False, scale_f16: bool = False):
        """Y [batch, rows] float64 = A [batch, cols] (bf16 bit patterns) times
        the transposed prefix-k weights (binary32 stage sums)."""
        A_bits = np.ascontiguousarray(np.atleast_2d(A_bits), dtype=np.uint16)
        batch = A_bits.shape[0]
        assert A_bits.shape[1] == cols
        sdt = np.uint16 if scale_f16 else np.float32
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=sdt) for a in scales[:k]]
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (ctypes.c_void_p * k)(*[a.ctypes.data for a in scales])
        zp = None
        if not sym:
            zeros = [np.ascontiguousarray(a, dtype=np.float32) for a in zeros[:k]]
            zp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in zeros])
        Y = np.zeros((batch, rows), np.float64)
        rc = self.lib.rrq_oracle_gemv(cp, sp, zp, rows, cols, group, k, int(sym), int(scale_f16),
                                      A_bits.ctypes.data_as(_u16p), batch,
                                      Y.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
        if rc != 0:
            raise ValueError("oracle rejected the product")
        return Y

    def prefill(self, codes, scales, zeros, rows: int, cols: int, group: int, k: int, A_bits,
                sym: bool = False, scale_f16: bool = False):
        """Y [tokens, rows] float64 = A [tokens, cols] (bf16 bit patterns) times
        the transposed bf16 prefix-k reconstruction, summed in binary64."""
        A_bits = np.ascontiguousarray(np.atleast_2d(A_bits), dtype=np.uint16)
        tokens = A_bits.shape[0]
        assert A_bits.shape[1] == cols
        sdt = np.uint16 if scale_f16 else np.float32
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=sdt) for a in scales[:k]]
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (ctypes.c_void_p * k)(*[a.ctypes.data for a in scales])
        zp = None
        if not sym:
            zeros = [np.ascontiguousarray(a, dtype=np.float32) for a in zeros[:k]]
            zp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in zeros])
        Y = np.zeros((tokens, rows), np.float64)
        rc = self.lib.rrq_oracle_prefill(cp, sp, zp, rows, cols, group, k, int(sym), int(scale_f16),
                                         A_bits.ctypes.data_as(_u16p), tokens,
                                         Y.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
        if rc != 0:
            raise ValueError("oracle rejected the prefill product")
        return Y

    # -- heterogeneous stage widths (asymmetric grid) ----------------------------
    def quantize_group_bits(self, x, bits):
        """(Q, scale, zero, resid) for one group with per-stage widths."""
        x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
        g, S = x.size, len(bits)
        b = (ctypes.c_int * S)(*bits)
        Q = np.zeros((S, g), np.uint8)
        s = np.zeros(S, np.float32)
        z = np.zeros(S, np.float32)
        r = np.zeros((S, g), np.float32)
        rc = self.lib.rrq_oracle_quantize_group_bits(
            x.ctypes.data_as(_f32p), g, S, b, Q.ctypes.data_as(_u8p), s.ctypes.data_as(_f32p),
            z.ctypes.data_as(_f32p), r.ctypes.data_as(_f32p))
        if rc != 0:
            raise ValueError("oracle rejected the group")
        return Q, s, z, r

    def quantize_bits(self, W_bits, group, bits):
        """(codes, scales, zeros) with stage k's codes packed at bits[k] bits."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        n, S = rows * cols, len(bits)
        codes = [np.zeros((n * b + 7) // 8, np.uint8) for b in bits]
        scales = [np.zeros(n // group, np.float32) for _ in bits]
        zeros = [np.zeros(n // group, np.float32) for _ in bits]
        cp = (_u8p * S)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * S)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * S)(*[a.ctypes.data_as(_f32p) for a in zeros])
        rc = self.lib.rrq_oracle_quantize_bits(W_bits.ctypes.data_as(_u16p), rows, cols, group, S,
                                               (ctypes.c_int * S)(*bits), cp, sp, zp)
        if rc != 0:
            raise ValueError("oracle rejected the matrix")
        return codes, scales, zeros

    def quantize_from_base_bits(self, W_bits, base, group, bits):
        """Algorithm 1 with a base checkpoint and per-stage widths: base =
        (codes0, scales0, zeros0) at width bits[0]; returns the package
        (codes, scales, zeros) with stage 0 the given base."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        n, S = rows * cols, len(bits)
        codes = [np.ascontiguousarray(base[0], dtype=np.uint8).copy()] + \
            [np.zeros((n * b + 7) // 8, np.uint8) for b in bits[1:]]
        scales = [np.ascontiguousarray(base[1], dtype=np.float32).copy()] + [np.zeros(n // group, np.float32)
                                                                              for _ in bits[1:]]
        zeros = [np.ascontiguousarray(base[2], dtype=np.float32).copy()] + [np.zeros(n // group, np.float32)
                                                                             for _ in bits[1:]]
        cp = (_u8p * S)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * S)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * S)(*[a.ctypes.data_as(_f32p) for a in zeros])
        b = (ctypes.c_int * S)(*bits)
        rc = self.lib.rrq_oracle_quantize_from_base_bits(W_bits.ctypes.data_as(_u16p), rows, cols, group, S, b,
                                                         cp, sp, zp)
        if rc != 0:
            raise ValueError("oracle rejected the base-checkpoint build with widths")
        return codes, scales, zeros

    def product_bits(self, codes, scales, zeros, rows, cols, group, k, bits, A_bits, bf16_weights: bool):
        """Y [tokens, rows] float64: activations (bf16 bit patterns) times the
        prefix-k weights of a package with per-stage widths, binary32 (decode
        form) or bf16-rounded (prefill form)."""
        A_bits = np.ascontiguousarray(np.atleast_2d(A_bits), dtype=np.uint16)
        tokens = A_bits.shape[0]
        assert A_bits.shape[1] == cols
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=np.float32) for a in scales[:k]]
        zeros = [np.ascontiguousarray(a, dtype=np.float32) for a in zeros[:k]]
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in zeros])
        b = (ctypes.c_int * k)(*list(bits)[:k])
        Y = np.zeros((tokens, rows), np.float64)
        rc = self.lib.rrq_oracle_product_bits(cp, sp, zp, rows, cols, group, k, b, A_bits.ctypes.data_as(_u16p),
                                              tokens, int(bf16_weights),
                                              Y.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
        if rc != 0:
            raise ValueError("oracle rejected the product with per-stage widths")
        return Y

    def reconstruct_bits(self, codes, scales, zeros, rows, cols, group, k, bits):
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=np.float32) for a in scales[:k]]
        zeros = [np.ascontiguousarray(a, dtype=np.float32) for a in zeros[:k]]
        out = np.zeros((rows, cols), np.uint16)
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in scales])
        zp = (_f32p * k)(*[a.ctypes.data_as(_f32p) for a in zeros])
        rc = self.lib.rrq_oracle_reconstruct_bits(cp, sp, zp, rows, cols, group, k,
                                                  (ctypes.c_int * k)(*bits[:k]), out.ctypes.data_as(_u16p))
        if rc != 0:
            raise ValueError("oracle rejected the reconstruction")
        return out

    def group_pmr(self, W_bits, group):
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        rows, cols = W_bits.shape
        out = np.zeros(rows * cols // group, np.float64)
        rc = self.lib.rrq_oracle_group_pmr(W_bits.ctypes.data_as(_u16p), rows, cols, group,
                                           out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
        if rc != 0:
            raise ValueError("oracle rejected the matrix")
        return out

    def reconstruct_sym(self, codes, scales, rows: int, cols: int, group: int, k: int,
                        scale_f16: bool = True):
        """bf16 bit patterns [rows, cols] of the prefix-k reconstruction of a
        symmetric package."""
        sdt = np.uint16 if scale_f16 else np.float32
        codes = [np.ascontiguousarray(c, dtype=np.uint8) for c in codes[:k]]
        scales = [np.ascontiguousarray(a, dtype=sdt) for a in scales[:k]]
        out = np.zeros((rows, cols), np.uint16)
        cp = (_u8p * k)(*[c.ctypes.data_as(_u8p) for c in codes])
        sp = (ctypes.c_void_p * k)(*[a.ctypes.data for a in scales])
        rc = self.lib.rrq_oracle_reconstruct_sym(cp, sp, rows, cols, group, k, int(scale_f16),
                                                 out.ctypes.data_as(_u16p))
        if rc != 0:
            raise ValueError("oracle rejected the reconstruction")
        return out


_default = None


def load() -> Oracle:
    """The committed oracle, built on first use."""
    global _default
    if _default is None:
        _default = Oracle(build())
    return _default


def quantize_group(x, n_stages: int = 4):
    return load().quantize_group(x, n_stages)


def quantize(W_bits, group: int = 128, n_stages: int = 4):
    return load().quantize(W_bits, group, n_stages)


def reconstruct(codes, scales, zeros, rows, cols, group, k):
    return load().reconstruct(codes, scales, zeros, rows, cols, group, k)


def quantize_sym(W_bits, group: int = 128, n_stages: int = 4, scale_f16: bool = True):
    return load().quantize_sym(W_bits, group, n_stages, scale_f16)


def reconstruct_sym(codes, scales, rows, cols, group, k, scale_f16: bool = True):
    return load().reconstruct_sym(codes, scales, rows, cols, group, k, scale_f16)


def gemv(codes, scales, zeros, rows, cols, group, k, A_bits, sym: bool = False, scale_f16: bool = False):
    return load().gemv(codes, scales, zeros, rows, cols, group, k, A_bits, sym, scale_f16)


def prefill(codes, scales, zeros, rows, cols, group, k, A_bits, sym: bool = False, scale_f16: bool = False):
    return load().prefill(codes, scales, zeros, rows, cols, group, k, A_bits, sym, scale_f16)


def quantize_bits(W_bits, group, bits):
    return load().quantize_bits(W_bits, group, bits)


def reconstruct_bits(codes, scales, zeros, rows, cols, group, k, bits):
    return load().reconstruct_bits(codes, scales, zeros, rows, cols, group, k, bits)


def quantize_from_base_bits(W_bits, base, group, bits):
    return load().quantize_from_base_bits(W_bits, base, group, bits)


def product_bits(codes, scales, zeros, rows, cols, group, k, bits, A_bits, bf16_weights: bool):
    return load().product_bits(codes, scales, zeros, rows, cols, group, k, bits, A_bits, bf16_weights)


def group_pmr(W_bits, group):
    return load().group_pmr(W_bits, group)


def quantize_from_base(W_bits, base, group: int = 128, n_stages: int = 4, sym: bool = False,
                       scale_f16: bool = False):
    return load().quantize_from_base(W_bits, base, group, n_stages, sym, scale_f16)
