"""The CPU oracle over many host cores: TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg (and its ``--impl reference`` arm) may use this module.  It adds no
arithmetic: every package and reconstruction it produces comes from the
single-threaded oracle in ``rrq_oracle.c`` (Section 3.1 Eq. 1-3, Section 3.2
Eq. 4-8, Algorithm 1), run unchanged in P worker processes.

Groups run along rows and every row of a matrix is independent (a group never
spans two rows), so the oracle applied to rows [r0, r1) of W gives exactly
the slice [r0, r1) of every output of the whole matrix: codes
[r0*cols/4, r1*cols/4), scales and zeros [r0*cols/g, r1*cols/g), bf16
prefixes [r0*cols, r1*cols).  A task is such a row range.

Data travels through shared memory: the caller copies W (and, for a parity
check, the device's package and prefixes) into a ``SharedRegion``; a worker
maps the region, runs the oracle on its rows and compares slice by slice, so
only small result records cross the process boundary.  The pool starts its
workers with ``spawn`` (never ``fork``), so it is safe to create after the
calling process has initialised CUDA.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import time
from dataclasses import dataclass, replace
from multiprocessing import shared_memory

import numpy as np

#: package formats of the oracle: asymmetric grid (binary32 scale and zero),
#: symmetric grid with binary32 or binary16 scales
FORMATS = ("asym", "sym32", "sym16")


class SharedRegion:
    """A block of shared memory that worker processes map by name."""

    def __init__(self, nbytes: int):
        self.nbytes = int(nbytes)
        self.shm = shared_memory.SharedMemory(create=True, size=max(1, self.nbytes))
        self.name = self.shm.name

    def array(self, offset: int, dtype, count: int) -> np.ndarray:
        return np.ndarray((int(count),), dtype=dtype, buffer=self.shm.buf, offset=int(offset))

    def address(self) -> int:
        """Host address of the region's first byte (for page registration)."""
        return self.array(0, np.uint8, 1).ctypes.data

    def close(self):
        if self.shm is not None:
            self.shm.close()
            self.shm.unlink()
            self.shm = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


class Layout:
    """Byte offsets of arrays packed one after another (64-byte aligned)."""

    def __init__(self):
        self.size = 0

    def take(self, nbytes: int) -> int:
        off = self.size
        self.size += (int(nbytes) + 63) // 64 * 64
        return off


@dataclass(frozen=True)
class Task:
    """One oracle job on rows [row0, row0 + rows) of a bf16 matrix held in a
    shared region.  Offsets are byte offsets of the WHOLE matrix's arrays in
    the region; -1 marks an array that is absent.

    codes/scales/zeros: the device's package, per stage (compared when
    ``check`` is true).  prefixes[j]: the device's bf16 prefix with j+1
    stages.  recon: (k, offset) pairs of single-prefix reconstructions.
    With ``check`` false the task only runs the oracle (timing)."""
    region: str
    label: str
    fmt: str
    group: int
    n_stages: int
    rows: int
    cols: int
    w: int
    row0: int = 0
    nrows: int = -1
    codes: tuple = ()
    scales: tuple = ()
    zeros: tuple = ()
    prefixes: tuple = ()
    recon: tuple = ()
    check: bool = True
    oracle_prefixes: int = 0   # prefixes to reconstruct when only timing

    def split(self, max_weights: int) -> list:
        """Row-range tasks of at most about max_weights weights each."""
        per = max(1, int(max_weights) // self.cols)
        return [replace(self, row0=r, nrows=min(per, self.rows - r)) for r in range(0, self.rows, per)]


# ---------------------------------------------------------------------------
# worker side
# ---------------------------------------------------------------------------
# A worker keeps its mapping of a region until it exits: callers create a few
# regions, reuse them, and close the pool before unlinking them.
_REGIONS: dict = {}


def _map(name: str) -> shared_memory.SharedMemory:
    shm = _REGIONS.get(name)
    if shm is None:
        shm = shared_memory.SharedMemory(name=name)
        _REGIONS[name] = shm
    return shm


def _view(shm, offset, dtype, start, count):
    itemsize = np.dtype(dtype).itemsize
    return np.ndarray((int(count),), dtype=dtype, buffer=shm.buf, offset=int(offset) + int(start) * itemsize)


def _first_difference(a: np.ndarray, b: np.ndarray, start: int) -> str:
    bad = np.nonzero(a != b)[0]
    i = int(bad[0])
    return f"{bad.size} differ, first at element {start + i}: device {a[i]!r} oracle {b[i]!r}"


def run_task(t: Task) -> dict:
    """Runs the oracle on one task; returns {label, weights, seconds,
    mismatches} (mismatches: human-readable lines, empty when every
    compared byte is equal)."""
    import oracle
    rows = t.rows - t.row0 if t.nrows < 0 else t.nrows
    n0, n = t.row0 * t.cols, rows * t.cols
    g0, ng = n0 // t.group, n // t.group
    shm = _map(t.region)
    W = _view(shm, t.w, np.uint16, n0, n).reshape(rows, t.cols)
    sym, f16 = t.fmt != "asym", t.fmt == "sym16"
    sdt = np.uint16 if f16 else np.uint32   # scale bits as stored
    t0 = time.perf_counter()
    if sym:
        codes, scales = oracle.quantize_sym(W, t.group, t.n_stages, f16)
        zeros = None
    else:
        codes, scales, zeros = oracle.quantize(W, t.group, t.n_stages)

    def recon(k):
        if sym:
            return oracle.reconstruct_sym(codes, scales, rows, t.cols, t.group, k, f16)
        return oracle.reconstruct(codes, scales, zeros, rows, t.cols, t.group, k)

    bad = []
    where = f"{t.label} rows {t.row0}..{t.row0 + rows - 1}"
    if not t.check:
        for k in range(1, t.oracle_prefixes + 1):
            recon(k)
        return {"label": t.label, "weights": n, "seconds": time.perf_counter() - t0, "mismatches": bad}
    for k, off in enumerate(t.codes):
        got = _view(shm, off, np.uint8, n0 // 4, n // 4)
        if not np.array_equal(got, codes[k]):
            bad.append(f"{where} stage {k} codes: " + _first_difference(got, codes[k], n0 // 4))
    for k, off in enumerate(t.scales):
        got, want = _view(shm, off, sdt, g0, ng), scales[k].view(sdt)
        if not np.array_equal(got, want):
            bad.append(f"{where} stage {k} scales: " + _first_difference(got, want, g0))
    for k, off in enumerate(t.zeros):
        got, want = _view(shm, off, np.uint32, g0, ng), zeros[k].view(np.uint32)
        if not np.array_equal(got, want):
            bad.append(f"{where} stage {k} zeros: " + _first_difference(got, want, g0))
    wanted = [(j + 1, off) for j, off in enumerate(t.prefixes)] + list(t.recon)
    for k, off in wanted:
        want = recon(k).reshape(-1)
        got = _view(shm, off, np.uint16, n0, n)
        if not np.array_equal(got, want):
            bad.append(f"{where} prefix {k}: " + _first_difference(got, want, n0))
    return {"label": t.label, "weights": n, "seconds": time.perf_counter() - t0, "mismatches": bad}


def _init_worker():
    import oracle
    oracle.load()


# ---------------------------------------------------------------------------
# caller side
# ---------------------------------------------------------------------------
class OraclePool:
    """P worker processes (spawned) that run oracle tasks.  A worker that
    dies makes every pending result raise (BrokenProcessPool) instead of
    waiting forever."""

    def __init__(self, processes: int | None = None):
        from concurrent.futures import ProcessPoolExecutor
        import oracle
        oracle.build()  # once, before the workers load it
        self.processes = int(processes or os.cpu_count() or 1)
        self.pool = ProcessPoolExecutor(self.processes, mp_context=mp.get_context("spawn"),
                                        initializer=_init_worker)

    def submit(self, tasks) -> list:
        """Futures of run_task(t) for every task (their .result() waits)."""
        return [self.pool.submit(run_task, t) for t in tasks]

    def run(self, tasks) -> list:
        return [f.result() for f in self.submit(tasks)]

    def close(self):
        if self.pool is not None:
            self.pool.shutdown(wait=True, cancel_futures=True)
            self.pool = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def host_description() -> dict:
    """Core count and CPU model of this host (lscpu's model name, else
    /proc/cpuinfo, else the platform string)."""
    import platform
    import subprocess
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if not model:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    if line.lower().startswith("model name"):
                        model = line.split(":", 1)[1].strip()
                        break
        except OSError:
            pass
    return {"cores": os.cpu_count(), "cpu_model": model or platform.processor() or platform.machine(),
            "machine": platform.machine()}
