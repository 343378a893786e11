"""Whole-workload parity: every output the device wrote, compared with the
CPU oracle run over all host cores (oracle.pool).

A workload is cut into units (a layer of a stack, one matrix of a sweep).
For each unit the device results are copied into a shared-memory slot and
the oracle re-derives them in row-range tasks on P worker processes, while
the next unit is copied into the other slot.  Nothing is sampled: every
code byte, scale, zero and bf16 prefix is compared."""
from __future__ import annotations

import time
from dataclasses import dataclass, field

import numpy as np
import torch

from oracle.pool import Layout, OraclePool, SharedRegion, Task, host_description

TASK_WEIGHTS = 1 << 23          # weights per oracle task (8 Mi)

#: one line per whole-workload check, printed in pytest's terminal summary
REPORT: list = []


@dataclass
class Entry:
    """One matrix of a unit: its input, the device package, the device's
    prefixes (prefixes[j] = prefix with j+1 stages) and single-prefix
    reconstructions recon[k] produced by `recon_fn`."""
    label: str
    W: torch.Tensor
    pkg: object
    prefixes: list = field(default_factory=list)


@dataclass
class Unit:
    entries: list
    recon_ks: tuple = ()        # prefixes the device reconstructs on demand
    recon_fn: object = None     # recon_fn(k) -> device tensors, one per entry


def _fmt_name(pkg) -> str:
    from paper_2608_04048_gb300 import binding
    if pkg.grid == binding.GRID_ASYM:
        return "asym"
    return "sym16" if pkg.scale_type == binding.SCALE_F16 else "sym32"


def _layout(unit: Unit) -> tuple:
    """Byte offsets of one unit's arrays in a slot, and the total size."""
    lay = Layout()
    offsets = []
    for e in unit.entries:
        p = e.pkg
        n = p.rows * p.cols
        esz = 2 if _fmt_name(p) == "sym16" else 4
        offsets.append({
            "w": lay.take(2 * n),
            "codes": [lay.take(n // 4) for _ in range(p.n_stages)],
            "scales": [lay.take(n // p.group * esz) for _ in range(p.n_stages)],
            "zeros": [lay.take(4 * n // p.group) for _ in p.zeros],
            "prefixes": [lay.take(2 * n) for _ in e.prefixes],
            "recon": [(k, lay.take(2 * n)) for k in unit.recon_ks],
        })
    return offsets, lay.size


class Slot:
    """Shared memory for one unit's device results at a time."""

    def __init__(self, nbytes: int):
        self.region = SharedRegion(nbytes)
        self.pending = []
        self.registered = False
        try:  # page-locked: device-to-host copies at full link speed
            rt = torch.cuda.cudart()
            self.registered = int(rt.cudaHostRegister(self.region.address(), nbytes, 0)) == 0
        except (AttributeError, RuntimeError, TypeError):
            self.registered = False

    def put(self, offset: int, t: torch.Tensor):
        nbytes = t.numel() * t.element_size()
        dst = torch.from_numpy(self.region.array(offset, np.uint8, nbytes))
        dst.copy_(t.contiguous().view(torch.uint8).reshape(-1))

    def fill(self, unit: Unit, check: bool = True) -> list:
        """Copies the unit's device results in; returns its oracle tasks."""
        tasks = []
        self.offsets, size = _layout(unit)
        assert size <= self.region.nbytes
        for e, off in zip(unit.entries, self.offsets):
            p = e.pkg
            self.put(off["w"], e.W)
            if check:
                for k in range(p.n_stages):
                    self.put(off["codes"][k], p.codes[k])
                    self.put(off["scales"][k], p.scales[k])
                for k, z in enumerate(p.zeros):
                    self.put(off["zeros"][k], z)
                for j, o in enumerate(e.prefixes):
                    self.put(off["prefixes"][j], o)
        if check and unit.recon_ks:
            for ki, k in enumerate(unit.recon_ks):
                outs = unit.recon_fn(k)
                torch.cuda.synchronize()
                for o, off in zip(outs, self.offsets):
                    self.put(off["recon"][ki][1], o)
        for e, off in zip(unit.entries, self.offsets):
            p = e.pkg
            t = Task(self.region.name, e.label, _fmt_name(p), p.group, p.n_stages, p.rows, p.cols, off["w"],
                     codes=tuple(off["codes"]) if check else (), scales=tuple(off["scales"]) if check else (),
                     zeros=tuple(off["zeros"]) if check else (), prefixes=tuple(off["prefixes"]) if check else (),
                     recon=tuple(off["recon"]) if check else (), check=check)
            tasks += t.split(TASK_WEIGHTS)
        return tasks

    def close(self):
        if self.registered:
            torch.cuda.cudart().cudaHostUnregister(self.region.address())
            self.registered = False
        self.region.close()


def check_units(name: str, units: list, pool: OraclePool, n_slots: int = 2) -> dict:
    """Checks every unit; returns a summary and appends it to REPORT.  The
    caller asserts that summary['mismatches'] is empty."""
    t0 = time.perf_counter()
    size = max(_layout(u)[1] for u in units)
    slots = [Slot(size) for _ in range(min(n_slots, len(units)))]
    weights, core_s, mismatches = 0, 0.0, []

    def drain(slot):
        nonlocal weights, core_s
        for r in slot.pending:
            res = r.result()
            weights += res["weights"]
            core_s += res["seconds"]
            mismatches.extend(res["mismatches"])
        slot.pending = []

    try:
        for i, unit in enumerate(units):
            slot = slots[i % len(slots)]
            drain(slot)
            slot.pending = pool.submit(slot.fill(unit))
        for slot in slots:
            drain(slot)
    finally:
        for slot in slots:
            slot.close()
    wall = time.perf_counter() - t0
    host = host_description()
    summary = {"workload": name, "weights": weights, "wall_s": round(wall, 1), "oracle_core_s": round(core_s, 1),
               "processes": pool.processes, "cores": host["cores"], "cpu_model": host["cpu_model"],
               "mismatches": mismatches[:20], "n_mismatch_lines": len(mismatches)}
    REPORT.append(f"{name}: {weights:,} weights, every output compared with the oracle: "
                  f"{'EQUAL' if not mismatches else f'{len(mismatches)} MISMATCH LINES'}; "
                  f"{wall:.1f} s wall, {core_s:.0f} oracle core-s on {pool.processes} processes "
                  f"({host['cores']} cores, {host['cpu_model']})")
    return summary
