"""Benchmark of the RRQ hot path on GB300: package construction (Algorithm 1)
and prefix reconstruction (Eq. 8, k = 1..4) over synthetic weight stacks
shaped like the paper's models.

Default workload: a Qwen3-8B-shaped linear stack (36 layers x {q,k,v,o,gate,
up,down}, 6.95e9 bf16 weights, Student-t(3) weights with 0.1% +-20 sigma
outliers per row, group 128, four 2-bit stages).  Other workloads
(--workload): single_4096, qwen3_8b_layer, sweep_8192 (four distributions x
groups 32/64/128/256) and qwen3_32b_stack.

One step = rrq_quantize_prefixes over every matrix of the workload: the
package and the bf16 reconstructions at k = 1, 2, 3, 4 of every matrix, from
one read of W.  The metric is bf16 weight bytes processed per second of step
time (GB/s).  The stacks' inputs are far larger than L2; the smaller
workloads flush L2 before every timed call.  The breakdown times the package
alone (rrq_quantize), every prefix from the package and each prefix by its
own call, with a roofline entry for each; on the stacks it also replays the
step's launches from one CUDA graph (`step_cuda_graph`) beside the eager
timing.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                    [--split] [--impl reference]

Under torchrun every rank builds and processes its own stack (independent
matrices, no data-path collective): weak scaling, value = all ranks' bytes /
max over ranks of the timed region.  With --split the ranks share ONE stack,
each taking a disjoint set of its matrices (strong scaling).  Rank 0 prints
one JSON line.

--impl reference times the CPU oracle (the plain C implementation in oracle/,
as it stands, in one process per host core over row ranges) on a bounded
sample of the same workload; it is the slow reference arm, not a target.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

GROUP = 128
STAGES = 4
KS = (1, 2, 3, 4)
WORKLOAD = "qwen3_8b_stack"
METRIC = "RRQ package construction GB/s of bf16 weights and % of HBM peak; s per 8B-shaped stack"
WORKLOAD_TEXT = {
    "qwen3_8b_stack": "qwen3_8b_stack: 36 layers x (q 4096x4096, k/v 1024x4096, o 4096x4096, gate/up "
                      "12288x4096, down 4096x12288), bf16, Student-t(3) std 0.02 + 0.1% +-0.4 outliers per "
                      "row, group 128 along the input dim, 4 x 2-bit stages",
    "qwen3_8b_layer": "qwen3_8b_layer: one layer of the 36-layer stack's shapes and distribution",
}


def alg_bytes_quantize(n: int, g: int = GROUP, S: int = STAGES) -> float:
    """Algorithmic bytes of one rrq_quantize over n weights: bf16 read once,
    S stages of 2-bit codes, fp32 scale and zero per group."""
    return 2.0 * n + S * (n / 4.0 + 8.0 * n / g)


def alg_bytes_prefixes(n: int, k: int, g: int = GROUP) -> float:
    """Algorithmic bytes of one rrq_reconstruct_prefixes: k code planes and
    metadata read once, k bf16 outputs written."""
    return 2.0 * k * n + k * (n / 4.0 + 8.0 * n / g)


def alg_bytes_quantize_sym16(n: int, g: int = GROUP, S: int = STAGES) -> float:
    """Symmetric package with binary16 scales: bf16 in, per stage n/4 code
    bytes and 2 n/g scale bytes out."""
    return n * (2 + S * (0.25 + 2.0 / g))


def alg_bytes_prefixes_sym16(n: int, k: int, g: int = GROUP) -> float:
    return n * (k * (0.25 + 2.0 / g) + 2 * k)


def time_sym_f16(mats, p_outs, specs, stream, reps: int = 3) -> dict:
    """The same stack in the paper's stored format (symmetric grid, binary16
    scales): rrq_quantize_ex, then rrq_reconstruct_ex of every prefix, each
    timed with CUDA events after one warm-up (breakdown context; the step
    above is the asymmetric binary32 package)."""
    from paper_2608_04048_gb300 import binding
    G, F16 = binding.GRID_SYM, binding.SCALE_F16
    pkgs = [binding.Package.empty(sp.rows, sp.cols, GROUP, STAGES, mats[0].device, G, F16) for sp in specs]
    q_items = binding.quantize_descs(mats, pkgs)
    r_items = binding.reconstruct_descs(pkgs, p_outs, len(KS))
    quant = lambda: binding.rrq_quantize_ex(mats, GROUP, STAGES, G, F16, pkgs, stream, q_items)
    recon = lambda: binding.rrq_reconstruct_ex(pkgs, len(KS), True, p_outs, stream, r_items)
    quant(); recon()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    ev[0].record(stream)
    for _ in range(reps):
        quant()
    ev[1].record(stream)
    for _ in range(reps):
        recon()
    ev[2].record(stream)
    torch.cuda.synchronize()
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout (symmetric format)")
    q_s = ev[0].elapsed_time(ev[1]) / reps / 1e3
    r_s = ev[1].elapsed_time(ev[2]) / reps / 1e3
    q_alg = sum(alg_bytes_quantize_sym16(sp.numel) for sp in specs)
    r_alg = sum(alg_bytes_prefixes_sym16(sp.numel, len(KS)) for sp in specs)
    hbm = measured_peaks()["hbm_gbs"]
    del pkgs
    return {"format": "symmetric grid, binary16 scales (rrq_quantize_ex / rrq_reconstruct_ex)",
            "quantize_s_per_stack": round(q_s, 6), "quantize_alg_gbs": round(q_alg / q_s / 1e9, 1),
            "quantize_frac_of_measured_hbm": round(q_alg / q_s / 1e9 / hbm, 4),
            "reconstruct_prefixes_k1to4_s": round(r_s, 6),
            "reconstruct_prefixes_alg_gbs": round(r_alg / r_s / 1e9, 1),
            "reconstruct_frac_of_measured_hbm": round(r_alg / r_s / 1e9 / hbm, 4),
            "step_bf16_gbs": round(2.0 * sum(sp.numel for sp in specs) / (q_s + r_s) / 1e9, 2)}


def time_from_base(mats, pkgs, specs, stream, reps: int = 3) -> dict:
    """Algorithm 1 from a base checkpoint on the same stack: each package's
    stage 0 (left by the timed step) is taken as the given base and stages
    1..3 are rebuilt by rrq_quantize_from_base (reads W and the base stage,
    writes three stages: the same 3.25 B/weight as the full build)."""
    from paper_2608_04048_gb300 import binding
    items = binding.quantize_descs(mats, pkgs)
    run = lambda: binding.rrq_quantize_from_base(mats, pkgs, stream, items)
    run()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        run()
    b.record(stream)
    torch.cuda.synchronize()
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout (from base)")
    t = a.elapsed_time(b) / reps / 1e3
    alg = sum(alg_bytes_quantize(sp.numel) for sp in specs)
    return {"call": "rrq_quantize_from_base (asymmetric, binary32), stage 0 given",
            "s_per_stack": round(t, 6), "alg_gbs": round(alg / t / 1e9, 1),
            "frac_of_measured_hbm": round(alg / t / 1e9 / measured_peaks()["hbm_gbs"], 4)}


def time_gemv(pkgs, specs, stream, batch: int = 1, reps: int = 5) -> dict:
    """Decode product over the whole stack (Appendix C): rrq_gemv of every
    matrix's package at prefix k = 1..4 with one activation row, timed with
    CUDA events.  Algorithmic bytes: the first k stages of the package
    (k x (1/4 + 8/g) B per weight), the bf16 activations and the fp32 output."""
    from paper_2608_04048_gb300 import binding
    dev = pkgs[0].codes[0].device
    gen = torch.Generator(device=dev).manual_seed(77)
    acts = [torch.randn((batch, sp.cols), generator=gen, device=dev).to(torch.bfloat16) for sp in specs]
    ys = [torch.empty((batch, sp.rows), dtype=torch.float32, device=dev) for sp in specs]
    hbm = measured_peaks()["hbm_gbs"]
    out = {"call": f"rrq_gemv over all {len(specs)} matrices, batch {batch} (asymmetric binary32 package)"}
    for k in KS:
        items = binding.gemv_descs(pkgs, acts, ys, k)
        run = lambda st=stream: binding.rrq_gemv(pkgs, acts, k, ys, st, items)
        run()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            run()
        b.record(stream)
        torch.cuda.synchronize()
        t = a.elapsed_time(b) / reps / 1e3
        alg = sum(sp.numel * k * (0.25 + 8.0 / GROUP) + 2 * batch * sp.cols + 4 * batch * sp.rows
                  for sp in specs)
        out[f"k{k}"] = {"s_per_stack": round(t, 6), "alg_gbs": round(alg / t / 1e9, 1),
                        "frac_of_measured_hbm": round(alg / t / 1e9 / hbm, 4),
                        "weights_per_s": round(sum(sp.numel for sp in specs) / t, 1),
                        "weight_row_products_per_s": round(sum(sp.numel for sp in specs) * batch / t, 1)}
        if batch == 1:  # the same call's launches replayed from a CUDA graph (no host work per pass)
            tg, err = graph_seconds(run, stream, reps)
            out[f"k{k}"]["cuda_graph"] = {"error": err} if tg is None else {
                "s_per_stack": round(tg, 6), "frac_of_measured_hbm": round(alg / tg / 1e9 / hbm, 4)}
    return out


def graph_seconds(run, stream, reps: int):
    """Seconds per pass of run(stream) replayed from one CUDA graph captured
    on a side stream (relaxed capture mode), after one untimed replay;
    (None, reason) if the capture is refused."""
    side = torch.cuda.Stream(device=stream.device)
    graph = torch.cuda.CUDAGraph()
    try:
        side.wait_stream(stream)
        with torch.cuda.graph(graph, stream=side, capture_error_mode="relaxed"):
            run(side)
    except Exception as e:  # reported in the breakdown, never a silent fallback
        return None, f"{type(e).__name__}: {e}"[:200]
    with torch.cuda.stream(side):
        graph.replay()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(side)
        for _ in range(reps):
            graph.replay()
        b.record(side)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps / 1e3, None


def time_prefill(pkgs, specs, stream, tokens: int = 2048, reps: int = 2) -> dict:
    """Prefill product over the whole stack (Appendix C's product for many
    activation rows, on the tensor cores): rrq_prefill of each layer's 7
    packages (one call per layer, buffers shared by the layers) with `tokens`
    activation rows, at prefix k = 1..4, timed with CUDA events.  Work: 2 x
    tokens x rows x cols flops per matrix, against the measured bf16 dense
    peak (burst: the calls are timed alone)."""
    from paper_2608_04048_gb300 import binding
    dev = pkgs[0].codes[0].device
    per = 7
    layers = [list(range(i, min(i + per, len(specs)))) for i in range(0, len(specs), per)]
    gen = torch.Generator(device=dev).manual_seed(78)
    acts = [torch.randn((tokens, specs[j].cols), generator=gen, device=dev).to(torch.bfloat16) for j in layers[0]]
    ys = [torch.empty((tokens, specs[j].rows), dtype=torch.float32, device=dev) for j in layers[0]]
    peaks = measured_peaks()
    peak = peaks["bf16_tflops"]
    flops = 2.0 * tokens * sum(sp.numel for sp in specs)
    out = {"call": f"rrq_prefill over all {len(specs)} matrices, {tokens} tokens, one call per layer "
                   "(asymmetric binary32 package)", "tokens": tokens, "peak_tflops": peak,
           "peak_source": f"{peaks['source']} dense bf16 (burst)"}
    for k in KS:
        items = [binding.gemv_descs([pkgs[j] for j in L], acts[:len(L)], ys[:len(L)], k) for L in layers]

        def run():
            for L, it in zip(layers, items):
                binding.rrq_prefill([pkgs[j] for j in L], acts[:len(L)], k, ys[:len(L)], stream, it)
        run()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            run()
        b.record(stream)
        torch.cuda.synchronize()
        t = a.elapsed_time(b) / reps / 1e3
        out[f"k{k}"] = {"s_per_stack": round(t, 6), "tflops": round(flops / t / 1e12, 1),
                        "frac_of_measured_bf16": round(flops / t / 1e12 / peak, 4)}
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout (prefill)")
    return out


def time_bits(mats, p_outs, specs, stream, bits, reps: int = 3) -> dict:
    """A heterogeneous-width package of the same stack (asymmetric grid,
    stage widths `bits`): rrq_quantize_ex and all-prefix rrq_reconstruct_ex,
    CUDA events after one warm-up.  Bytes: 2 + sum_k (b_k/8 + 8/g) per weight
    to build; sum_k (b_k/8 + 8/g) + 2 S to reconstruct every prefix."""
    from paper_2608_04048_gb300 import binding
    S = len(bits)
    pkgs = [binding.Package.empty(sp.rows, sp.cols, GROUP, S, mats[0].device, binding.GRID_ASYM,
                                  binding.SCALE_F32, list(bits)) for sp in specs]
    q_items = binding.quantize_descs(mats, pkgs)
    outs = [o[:S] for o in p_outs]
    r_items = binding.reconstruct_descs(pkgs, outs, S)
    quant = lambda: binding.rrq_quantize_ex(mats, GROUP, S, binding.GRID_ASYM, binding.SCALE_F32,
                                            pkgs, stream, q_items, bits=list(bits))
    recon = lambda: binding.rrq_reconstruct_ex(pkgs, S, True, outs, stream, r_items)
    quant(); recon()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    ev[0].record(stream)
    for _ in range(reps):
        quant()
    ev[1].record(stream)
    for _ in range(reps):
        recon()
    ev[2].record(stream)
    torch.cuda.synchronize()
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout (widths)")
    q_s = ev[0].elapsed_time(ev[1]) / reps / 1e3
    r_s = ev[1].elapsed_time(ev[2]) / reps / 1e3
    per = sum(b / 8 + 8.0 / GROUP for b in bits)
    n = sum(sp.numel for sp in specs)
    hbm = measured_peaks()["hbm_gbs"]
    del pkgs
    return {"quantize_s_per_stack": round(q_s, 6), "quantize_alg_gbs": round(n * (2 + per) / q_s / 1e9, 1),
            "quantize_frac_of_measured_hbm": round(n * (2 + per) / q_s / 1e9 / hbm, 4),
            "reconstruct_prefixes_s": round(r_s, 6),
            "reconstruct_prefixes_alg_gbs": round(n * (per + 2 * S) / r_s / 1e9, 1),
            "reconstruct_frac_of_measured_hbm": round(n * (per + 2 * S) / r_s / 1e9 / hbm, 4)}


def time_pmr(mats, specs, stream, reps: int = 5) -> dict:
    """rrq_group_pmr over the stack (2 B per weight read, 4 B per group
    written)."""
    from paper_2608_04048_gb300 import binding
    binding.rrq_group_pmr(mats, GROUP, stream)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        binding.rrq_group_pmr(mats, GROUP, stream)
    b.record(stream)
    torch.cuda.synchronize()
    t = a.elapsed_time(b) / reps / 1e3
    n = sum(sp.numel for sp in specs)
    alg = n * (2 + 4.0 / GROUP)
    return {"s_per_stack": round(t, 6), "alg_gbs": round(alg / t / 1e9, 1),
            "frac_of_measured_hbm": round(alg / t / 1e9 / measured_peaks()["hbm_gbs"], 4)}


def alg_bytes_reconstruct(n: int, k: int, g: int = GROUP) -> float:
    """Algorithmic bytes of one rrq_reconstruct at prefix k: k code planes and
    metadata read, bf16 written."""
    return 2.0 * n + k * (n / 4.0 + 8.0 * n / g)


def measured_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d.get("bf16_tflops") or 1900.0),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.device_index = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.device_index}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict:
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for name, val in zip(names, parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        # samples under load: the upper half of the clock distribution is
        # not needed; report the median of all samples taken in the region
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# distributed helpers (one process per GPU, launched by torchrun)
# ---------------------------------------------------------------------------
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def shard_seed_offset(rank: int) -> int:
    """Each rank builds its own stack of independent matrices: seeds shifted
    by a per-rank offset far above the stack's own seed range."""
    return 1_000_003 * rank


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------
L2_BYTES = 126 * 2**20
FLUSH_WORKLOADS = ("single_4096", "qwen3_8b_layer", "sweep_8192")   # inputs near or below L2


def shard_matrices(specs, world: int, rank: int) -> list:
    """Indices of the matrices rank `rank` takes when one stack is split over
    `world` ranks: largest first, each to the rank with the fewest weights so
    far (ties to the lower rank); every matrix goes to exactly one rank."""
    load = [0] * world
    owner = {}
    for i in sorted(range(len(specs)), key=lambda i: (-specs[i].numel, i)):
        r = min(range(world), key=lambda j: (load[j], j))
        owner[i] = r
        load[r] += specs[i].numel
    return [i for i in range(len(specs)) if owner[i] == rank]


class L2Flush:
    """Writes a buffer twice the size of L2 (between timed calls of
    workloads whose inputs would otherwise stay resident)."""

    def __init__(self, device):
        self.buf = torch.empty(2 * L2_BYTES // 4, dtype=torch.int32, device=device)
        self.n = 0

    def __call__(self):
        self.n += 1
        self.buf.fill_(self.n)


def time_graph(wl, calls, reps: int):
    """Seconds per pass of `calls` (the workload's calls, which launch on
    wl.stream) replayed from one CUDA graph; see graph_seconds."""
    old = wl.stream

    def run(side):
        wl.stream = side
        try:
            for c in calls:
                c()
        finally:
            wl.stream = old
    return graph_seconds(run, old, reps)


def time_calls(calls, stream, reps: int, flush=None) -> float:
    """Mean seconds of one pass over `calls` (after one untimed pass).
    With `flush`, L2 is flushed before every call and only the calls are
    timed (CUDA events around each); otherwise one event pair brackets the
    passes."""
    for c in calls:
        c()
    if flush is None:
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            for c in calls:
                c()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps / 1e3
    evs = []
    for _ in range(reps):
        for c in calls:
            flush()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            c()
            b.record(stream)
            evs.append((a, b))
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs) / reps / 1e3


class Workload:
    """The device side of one named workload: inputs, packages, prefix
    outputs, and the calls that make up a step and its breakdown parts.

    The calls group matrices that share a group size.  If every matrix's
    four bf16 prefixes fit in HBM beside the stack they get their own
    outputs; otherwise (the Qwen3-32B-shaped stack) the matrices go in
    layers of 7 that write their prefixes into one set of buffers, reused
    by every layer."""

    def __init__(self, specs, device, seed_offset: int, stream):
        from paper_2608_04048_gb300 import binding, workloads
        self.specs, self.stream, self.device = specs, stream, device
        self.n_total = sum(sp.numel for sp in specs)
        cache = {}
        self.mats = []
        for sp in specs:  # the sweep's group sizes share one input per distribution
            key = (sp.rows, sp.cols, sp.seed, sp.dist)
            if key not in cache:
                cache[key] = workloads.generate(sp.rows, sp.cols, sp.seed + seed_offset, sp.dist, device)
            self.mats.append(cache[key])
        self.pkgs = [binding.Package.empty(sp.rows, sp.cols, sp.group, STAGES, device) for sp in specs]
        pkg_bytes = sum(p.nbytes() for p in self.pkgs)
        free, _ = torch.cuda.mem_get_info(device)
        own = len(KS) * 2 * self.n_total
        self.own_outputs = own + 4 * 2**30 < free
        # units: matrices that go together in one call (same group; a layer
        # of 7 when the outputs are shared)
        per = None if self.own_outputs else 7
        self.units = []
        for g in sorted({sp.group for sp in specs}):
            idx = [i for i, sp in enumerate(specs) if sp.group == g]
            if per is None:
                self.units.append(idx)
            else:
                self.units += [idx[i:i + per] for i in range(0, len(idx), per)]
        if self.own_outputs:
            self.p_outs = [[torch.empty((sp.rows, sp.cols), dtype=torch.bfloat16, device=device) for _ in KS]
                           for sp in specs]
        else:
            shared = [[torch.empty((specs[i].rows, specs[i].cols), dtype=torch.bfloat16, device=device) for _ in KS]
                      for i in self.units[0]]
            self.p_outs = [shared[j % len(shared)] for j in range(len(specs))]
            for u in self.units:
                assert all((specs[i].rows, specs[i].cols) == (specs[self.units[0][j]].rows,
                                                              specs[self.units[0][j]].cols)
                           for j, i in enumerate(u))
        self.pkg_bytes = pkg_bytes

    def group_of(self, unit) -> int:
        return self.specs[unit[0]].group

    def step_calls(self):
        """rrq_quantize_prefixes per unit: the package and every prefix."""
        from paper_2608_04048_gb300 import binding
        calls = []
        for u in self.units:
            mats, pkgs, outs = [self.mats[i] for i in u], [self.pkgs[i] for i in u], [self.p_outs[i] for i in u]
            items = binding.quantize_prefixes_descs(mats, pkgs, outs)
            g = self.group_of(u)
            calls.append(lambda mats=mats, pkgs=pkgs, outs=outs, items=items, g=g: binding.rrq_quantize_prefixes(
                mats, g, STAGES, binding.GRID_ASYM, binding.SCALE_F32, pkgs, outs, self.stream, items))
        return calls

    def quantize_calls(self):
        """rrq_quantize_batch per group size (the package only, Algorithm 1)."""
        from paper_2608_04048_gb300 import binding
        calls = []
        for g in sorted({sp.group for sp in self.specs}):
            idx = [i for i, sp in enumerate(self.specs) if sp.group == g]
            mats, pkgs = [self.mats[i] for i in idx], [self.pkgs[i] for i in idx]
            items = binding.quantize_items(mats, pkgs)
            calls.append(lambda mats=mats, pkgs=pkgs, items=items, g=g: binding.rrq_quantize_batch(
                mats, pkgs, g, STAGES, stream=self.stream, items=items))
        return calls

    def reconstruct_calls(self, k: int | None):
        """rrq_reconstruct_batch at prefix k (k given) or
        rrq_reconstruct_prefixes_batch of every prefix (k None), per unit."""
        from paper_2608_04048_gb300 import binding
        calls = []
        for u in self.units:
            pkgs, outs = [self.pkgs[i] for i in u], [self.p_outs[i] for i in u]
            if k is None:
                items = binding.prefixes_items(pkgs, outs, len(KS))
                calls.append(lambda pkgs=pkgs, outs=outs, items=items: binding.rrq_reconstruct_prefixes_batch(
                    pkgs, len(KS), outs, stream=self.stream, items=items))
            else:
                one = [o[k - 1] for o in outs]
                items = binding.reconstruct_items(pkgs, one)
                calls.append(lambda pkgs=pkgs, one=one, items=items, k=k: binding.rrq_reconstruct_batch(
                    pkgs, k, one, stream=self.stream, items=items))
        return calls


def roofline_entry(kernel: str, alg_bytes: float, seconds: float, peak: float, launches: int,
                   traffic_key: str | None) -> dict:
    achieved = alg_bytes / seconds / 1e9
    traffic = recorded_traffic(traffic_key, alg_bytes / launches, alg_bytes / launches) if traffic_key else None
    return {"kernel": kernel, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
            "frac": round(achieved / peak, 4), "frac_of_nominal_8tbs": round(achieved / 8000.0, 4),
            "alg_bytes_per_launch": round(alg_bytes / launches), "s_per_pass": round(seconds, 6),
            "traffic": traffic}


def run_gpu(args, world, rank, local) -> dict | None:
    from paper_2608_04048_gb300 import binding, build, workloads
    build.build()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    specs_all = workloads.config_matrices(args.workload)
    if args.split:  # one stack over all ranks (strong scaling)
        specs = [specs_all[i] for i in shard_matrices(specs_all, world, rank)]
        seed_offset = 0
    else:           # a stack per rank (weak scaling)
        specs = specs_all
        seed_offset = shard_seed_offset(rank)
    stream = torch.cuda.current_stream(device)
    binding.rrq_get_device_status()
    wl = Workload(specs, device, seed_offset, stream)
    n_total = wl.n_total
    flush = L2Flush(device) if args.workload in FLUSH_WORKLOADS else None
    steps_calls = wl.step_calls()

    def step():
        for c in steps_calls:
            if flush is not None:
                flush()
            c()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout during warm-up")

    # the timed region: events around every call when L2 is flushed between
    # calls (the flushes are not timed), else around each step
    per_call = flush is not None
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in (steps_calls if per_call else [None])] for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for s in range(args.steps):
            if per_call:
                for (a, b), c in zip(ev[s], steps_calls):
                    flush()
                    a.record(stream)
                    c()
                    b.record(stream)
            else:
                a, b = ev[s][0]
                a.record(stream)
                step()
                b.record(stream)
        t1.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    status = binding.rrq_get_device_status()
    if status != 0:
        raise RuntimeError(f"kernel status {status} in the timed region")
    f_ms = [sum(a.elapsed_time(b) for a, b in evs) for evs in ev]
    elapsed_ms = sum(f_ms) if per_call else t0.elapsed_time(t1)
    elapsed_ms = max_over_ranks(elapsed_ms, world)

    # breakdown: the package alone (rrq_quantize), every prefix from the
    # package, and each prefix by its own call
    q_calls = wl.quantize_calls()
    q_s = time_calls(q_calls, stream, 3, flush)
    groups = sorted({sp.group for sp in specs})
    q_by_group = {g: time_calls([c], stream, 3, flush) for g, c in zip(groups, q_calls)} if len(groups) > 1 else None
    r_s = time_calls(wl.reconstruct_calls(None), stream, 3, flush)
    each_k = {k: time_calls(wl.reconstruct_calls(k), stream, 2, flush) for k in KS}
    # the step's launches replayed from a CUDA graph (stacks: no L2 flush
    # between calls), beside the eager timing above
    graph_s, graph_err = time_graph(wl, steps_calls, args.steps) if flush is None else (None, None)
    torch.cuda.synchronize()
    if binding.rrq_get_device_status() != 0:
        raise RuntimeError("a kernel reported a timeout in the breakdown")

    stack = args.workload == "qwen3_8b_stack" and wl.own_outputs and not args.no_sym
    # the symmetric binary16 format and the two products also on one layer
    # (the size their ncu captures take)
    products = stack or (args.workload == "qwen3_8b_layer" and wl.own_outputs and not args.no_sym)
    mats, pkgs, p_outs = wl.mats, wl.pkgs, wl.p_outs
    sym = time_sym_f16(mats, p_outs, specs, stream) if products else None
    from_base = time_from_base(mats, pkgs, specs, stream) if stack else None
    gemv = time_gemv(pkgs, specs, stream) if products else None
    batches = [int(x) for x in args.gemv_batches.split(",") if x.strip()]
    gemv_batches = {f"batch{b}": time_gemv(pkgs, specs, stream, batch=b) for b in batches if b != 1} \
        if products and any(b != 1 for b in batches) else None
    prefill = time_prefill(pkgs, specs, stream) if products else None
    bits = {"+".join(map(str, b)): time_bits(mats, p_outs, specs, stream, b) for b in ((1, 3), (3, 1))} \
        if stack else None
    pmr = time_pmr(mats, specs, stream) if stack else None
    e2e = run_e2e(args, mats, pkgs, p_outs, specs, stream, world) \
        if not args.no_e2e and wl.own_outputs and len(wl.units) == 1 else None
    if rank != 0:
        return None

    peaks = measured_peaks()
    hbm = peaks["hbm_gbs"]
    clock_summary = clocks.summary()
    step_s = elapsed_ms / 1e3 / args.steps
    bytes_bf16 = 2.0 * n_total
    total_bf16 = 2.0 * sum(sp.numel for sp in specs_all) if args.split else world * bytes_bf16
    value = total_bf16 / step_s / 1e9
    f_s = statistics.mean(f_ms) / 1e3
    g_of = lambda sp: sp.group
    f_alg = sum(alg_bytes_quantize(sp.numel, g_of(sp)) + STAGES * 2 * sp.numel for sp in specs)
    q_alg = sum(alg_bytes_quantize(sp.numel, g_of(sp)) for sp in specs)
    r_alg = sum(alg_bytes_prefixes(sp.numel, len(KS), g_of(sp)) for sp in specs)
    k_alg = {k: sum(alg_bytes_reconstruct(sp.numel, k, g_of(sp)) for sp in specs) for k in KS}
    per_launch = 64  # matrices per kernel launch of the batch entry points
    launches = sum(math.ceil(len(u) / per_launch) for u in wl.units)
    q_launches = sum(math.ceil(sum(1 for sp in specs if sp.group == g) / per_launch)
                     for g in {sp.group for sp in specs})
    traffic = recorded_traffic("rrq_quantize_prefixes", f_alg / launches, f_alg / launches) \
        if args.workload in TRAFFIC_WORKLOADS else None
    rooflines = {
        "rrq_quantize": roofline_entry("quantize_tile_kernel<g,0,64> (n % 64 == 0; else quantize_kernel<g,0,0>): "
                                       "rrq_quantize_batch, the package only", q_alg, q_s,
                                       hbm, q_launches,
                                       "rrq_quantize" if args.workload in TRAFFIC_WORKLOADS else None),
        "rrq_reconstruct_prefixes": roofline_entry(
            "reconstruct_kernel<g,4,1,0>: rrq_reconstruct_prefixes_batch, every prefix 1..4 from the package",
            r_alg, r_s, hbm, launches, "rrq_reconstruct_prefixes" if args.workload in TRAFFIC_WORKLOADS else None),
    }
    for k in KS:
        rooflines[f"rrq_reconstruct_k{k}"] = roofline_entry(
            f"reconstruct_tile_kernel<g,{k},0> (whole 2048-weight chunks; else reconstruct_kernel<g,{k},0,0>): "
            f"rrq_reconstruct_batch at prefix k={k}", k_alg[k], each_k[k], hbm, launches,
            "rrq_reconstruct_k4" if k == 4 and args.workload in TRAFFIC_WORKLOADS else None)
    l2_text = (f"L2 flushed ({2 * L2_BYTES // 2**20} MiB write) before every timed call" if flush is not None else
               f"inputs {2 * n_total / 1e9:.2f} GB per rank, larger than the {L2_BYTES // 2**20} MiB L2; no flush")
    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(elapsed_ms / args.steps, 3),
        "higher_is_better": True,
        "scaling": "strong" if args.split else "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {
            "workload": WORKLOAD_TEXT.get(args.workload, args.workload),
            "step": (f"rrq_quantize_prefixes on all {len(specs)} matrices ({len(steps_calls)} call(s)): the "
                     f"package and the k=1,2,3,4 bf16 reconstructions of every matrix in one pass"
                     + ("" if wl.own_outputs else "; the prefixes of each layer of 7 go to one set of "
                        "buffers reused by every layer (the four prefixes of the stack do not fit in HBM)")),
            "weights_per_rank": n_total,
            "l2": l2_text,
            "parallelism": (f"one stack split over {world} rank(s) by matrices (largest first to the least "
                            f"loaded rank)" if args.split else f"{world} independent rank(s), one stack each"),
        },
        "breakdown": {
            "step_alg_gbs": round(f_alg / f_s / 1e9, 1),
            "step_cuda_graph": None if flush is not None else (
                {"error": graph_err} if graph_s is None else {
                    "ms_per_step": round(graph_s * 1e3, 3),
                    "bf16_gbs": round(bytes_bf16 / graph_s / 1e9, 2),
                    "frac_of_measured_hbm": round(f_alg / graph_s / 1e9 / hbm, 4),
                    "api_calls_per_step": len(steps_calls),
                    "kernel_launches_per_step": launches,
                    "eager_ms_per_step": round(elapsed_ms / args.steps, 3)}),
            "step_frac_of_measured_hbm": round(f_alg / f_s / 1e9 / hbm, 4),
            "two_calls_s_per_stack": round(q_s + r_s, 6),
            "two_calls_bf16_gbs": round(bytes_bf16 / (q_s + r_s) / 1e9, 2),
            "quantize_s_per_stack": round(q_s, 6),
            "quantize_alg_gbs": round(q_alg / q_s / 1e9, 1),
            "quantize_bf16_in_gbs": round(bytes_bf16 / q_s / 1e9, 1),
            "quantize_weights_per_s": round(n_total / q_s, 1),
            "quantize_frac_of_measured_hbm": round(q_alg / q_s / 1e9 / hbm, 4),
            "quantize_frac_of_nominal_8tbs": round(q_alg / q_s / 1e9 / 8000.0, 4),
            "reconstruct_prefixes_k1to4_s": round(r_s, 6),
            "reconstruct_prefixes_alg_gbs": round(r_alg / r_s / 1e9, 1),
            "reconstruct_frac_of_measured_hbm": round(r_alg / r_s / 1e9 / hbm, 4),
            "reconstruct_separate_k1to4_s": round(sum(each_k.values()), 6),
            "reconstruct_separate_alg_gbs": round(sum(k_alg.values()) / sum(each_k.values()) / 1e9, 1),
            "quantize_by_group": None if q_by_group is None else {
                f"g{g}": {"s": round(t, 6), "alg_gbs": round(a / t / 1e9, 1), "frac_of_measured_hbm": round(a / t / 1e9 / hbm, 4),
                          "frac_of_nominal_8tbs": round(a / t / 1e9 / 8000.0, 4)}
                for g, t in q_by_group.items()
                for a in [sum(alg_bytes_quantize(sp.numel, g) for sp in specs if sp.group == g)]},
            "paper_context_s": {"full_all_rtn_package_qwen3_8b_a100": 1293, "four_rtn_passes_a100": 412},
            "sym_f16": sym,
            "from_base": from_base,
            "gemv_decode": gemv,
            "gemv_decode_batches": gemv_batches,
            "prefill": prefill,
            "widths": bits,
            "group_pmr": pmr,
        },
        "roofline": {"kernel": "rrq_quantize_prefixes (quantize_kernel, build with prefixes)",
                     "bound": "hbm", "achieved": round(f_alg / f_s / 1e9, 1), "peak": hbm,
                     "peak_source": f"{peaks['source']} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                     "unit": "GB/s", "frac": round(f_alg / f_s / 1e9 / hbm, 4),
                     "alg_bytes_per_weight": round(f_alg / n_total, 4), "traffic": traffic},
        "rooflines": rooflines,
        "clocks": clock_summary,
        "gpu_launches": launches * args.steps,
        "e2e": e2e,
    }
    if args.cpu_seconds > 0 and world == 1:  # the host's cores, once (rank 0 at N=1)
        samples = [(specs[i].name, wl.mats[i]) for i in range(len(specs))]
        line["cpu_baseline"] = cpu_baseline(samples, args.cpu_seconds)
    return line


# workloads whose DRAM traffic per algorithmic byte the committed ncu capture
# (one Qwen3-8B-shaped layer) represents: the same shapes and group size
TRAFFIC_WORKLOADS = ("qwen3_8b_stack", "qwen3_8b_layer")


def recorded_traffic(kernel: str, q_bytes_per_launch: float, r_bytes_per_launch: float):
    """DRAM bytes per launch of `kernel` from the committed ncu summary
    (profiles/traffic.json), scaled to this workload's average launch by the
    ratio of DRAM to algorithmic bytes measured there; None when the kernel
    source changed since the capture."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f)
    entry = rec.get(kernel)
    if not entry or kernel not in KERNEL_SOURCES or entry.get("source_sha256") != kernel_source_hash(kernel):
        return None
    per_alg = entry["dram_bytes"] / entry["alg_bytes"]
    alg = r_bytes_per_launch if kernel == "rrq_reconstruct_prefixes" else q_bytes_per_launch
    return round(per_alg * alg)


# the source files each recorded kernel is compiled from
KERNEL_SOURCES = {
    "rrq_quantize": ["quantize_tile_kernel.cuh", "quantize_kernel.cuh", "quantize.cu"],
    "rrq_quantize_ex_sym_f16": ["quantize_tile_kernel.cuh", "quantize_kernel.cuh", "quantize.cu"],
    "rrq_reconstruct_prefixes": ["reconstruct_kernel.cuh", "reconstruct_tile_kernel.cuh", "reconstruct_asym_f32.cu"],
    "rrq_reconstruct_k4": ["reconstruct_kernel.cuh", "reconstruct_tile_kernel.cuh", "reconstruct_asym_f32.cu"],
    "rrq_reconstruct_ex_sym_f16": ["reconstruct_kernel.cuh", "reconstruct_tile_kernel.cuh", "reconstruct_sym_f16.cu"],
    "rrq_quantize_prefixes": ["quantize_kernel.cuh", "quantize_emit.cu"],
    "rrq_gemv_k1": ["gemv_mma_kernel.cuh", "gemv_kernel.cuh", "gemv_mma_asym_f32.cu", "gemv_asym_f32.cu"],
    "rrq_gemv_k4": ["gemv_mma_kernel.cuh", "gemv_kernel.cuh", "gemv_mma_asym_f32.cu", "gemv_asym_f32.cu"],
}

# the kernel (ncu demangled-name prefix) and algorithmic bytes per weight at
# group 128 behind each recorded entry
TRAFFIC_KERNELS = {
    "rrq_quantize": ("quantize_tile_kernel<128, 0,", 3.25),
    "rrq_quantize_ex_sym_f16": ("quantize_tile_kernel<128, 2,", 2 + 4 * (0.25 + 2 / 128)),
    "rrq_reconstruct_prefixes": ("reconstruct_kernel<128, 4, 1, 0>", 9.25),
    "rrq_reconstruct_k4": ("reconstruct_tile_kernel<128, 4, 0>", 3.25),
    "rrq_quantize_prefixes": ("quantize_kernel<128, 0, 2>", 11.25),
    "rrq_reconstruct_ex_sym_f16": ("reconstruct_kernel<128, 4, 1, 2>", 4 * (0.25 + 2 / 128) + 8),
    "rrq_gemv_k1": ("gemv_mma_kernel<0, 1, 128,", 0.25 + 8 / 128),
    "rrq_gemv_k4": ("gemv_mma_kernel<0, 4, 128,", 4 * (0.25 + 8 / 128)),
}


def record_traffic(csv_path: str, workload: str = "qwen3_8b_layer"):
    """Writes profiles/traffic.json from an ncu CSV (--metrics
    dram__bytes_read.sum,dram__bytes_write.sum --csv --log-file) of a bench.py
    run on `workload`: for each recorded kernel its first launch's DRAM bytes,
    the algorithmic bytes of one launch over the workload, and the SHA-256 of
    its sources."""
    import csv
    from paper_2608_04048_gb300 import workloads
    n = sum(sp.numel for sp in workloads.config_matrices(workload))
    rows = list(csv.DictReader(line for line in open(csv_path) if line.startswith('"')))
    launches = {}
    for r in rows:
        key = (r["ID"], r["Kernel Name"])
        launches.setdefault(key, {})[r["Metric Name"]] = (float(r["Metric Value"].replace(",", "")), r["Metric Unit"])
    unit = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9}
    path = os.path.join(ROOT, "profiles", "traffic.json")
    rec = json.load(open(path)) if os.path.exists(path) else {}
    for name, (prefix, per_weight) in TRAFFIC_KERNELS.items():
        for (lid, kname), m in sorted(launches.items(), key=lambda x: int(x[0][0])):
            if prefix in kname:
                dram = sum(v * unit[u] for k, (v, u) in m.items() if k in ("dram__bytes_read.sum", "dram__bytes_write.sum"))
                rec[name] = {"dram_bytes": int(dram), "alg_bytes": int(per_weight * n),
                             "capture": f"{kname.split('(rrq')[0].replace('void rrq::<unnamed>::', '').strip()}: "
                                        f"launch {lid} of bench.py --workload "
                                        f"{workload} ({n:,} weights), ncu dram__bytes_read.sum + dram__bytes_write.sum",
                             "source_sha256": kernel_source_hash(name),
                             "dram_over_alg": round(dram / (per_weight * n), 4)}
                break
    with open(path, "w") as f:
        json.dump(rec, f, indent=1)
        f.write("\n")


def kernel_source_hash(kernel: str) -> str:
    """SHA-256 over the sources of one kernel (its own files plus the shared
    device helpers and the host/device interface header)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_04048_gb300", "csrc")
    for name in KERNEL_SOURCES[kernel] + ["rrq_device.cuh", "rrq_internal.h"]:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode())
            h.update(f.read())
    return h.hexdigest()


def run_e2e(args, mats, pkgs, p_outs, specs, stream, world) -> dict:
    """Same metric through the public API with host buffers: every step copies
    each matrix from pinned host memory to the device, builds its package and
    its k=1..4 reconstructions (rrq_quantize_prefixes), and copies the package
    and every reconstruction back to pinned host buffers, all inside the timed
    region.  Layers are pipelined over three streams (copy in, build, copy
    out); the timed region ends when every stream is done."""
    from paper_2608_04048_gb300 import binding
    def pinned_like(t):
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h
    host_W = [pinned_like(W) for W in mats]
    host_pkg = [[torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in p.codes + p.scales + p.zeros]
                for p in pkgs]
    max_n = max(sp.numel for sp in specs)
    host_out = torch.empty(max_n, dtype=torch.bfloat16).pin_memory()
    h2d = sum(W.numel() * 2 for W in mats)
    d2h = sum(t.numel() * t.element_size() for p in host_pkg for t in p) + \
        len(KS) * sum(sp.numel * 2 for sp in specs)

    # one layer (7 matrices) per chunk, on three streams: the copy in of chunk
    # i+1 and the copy out of chunk i-1 overlap the build of chunk i
    per = 7
    chunks = [list(range(i, min(i + per, len(mats)))) for i in range(0, len(mats), per)]
    c_items = [binding.quantize_prefixes_descs([mats[j] for j in L], [pkgs[j] for j in L], [p_outs[j] for j in L])
               for L in chunks]
    dev = mats[0].device
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev = lambda: [torch.cuda.Event() for _ in chunks]
    ev_in, ev_built, ev_out = ev(), ev(), ev()
    started = [False]

    def step():
        for ci, L in enumerate(chunks):
            with torch.cuda.stream(s_in):
                if started[0]:  # the previous step's build of this chunk has read W
                    s_in.wait_event(ev_built[ci])
                for j in L:
                    mats[j].copy_(host_W[j], non_blocking=True)
                ev_in[ci].record(s_in)
            stream.wait_event(ev_in[ci])
            if started[0]:  # the previous step's copy out of this chunk is done
                stream.wait_event(ev_out[ci])
            binding.rrq_quantize_prefixes([mats[j] for j in L], GROUP, STAGES, binding.GRID_ASYM,
                                          binding.SCALE_F32, [pkgs[j] for j in L], [p_outs[j] for j in L],
                                          stream, c_items[ci])
            ev_built[ci].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_built[ci])
                for j in L:
                    for h, d in zip(host_pkg[j], pkgs[j].codes + pkgs[j].scales + pkgs[j].zeros):
                        h.copy_(d, non_blocking=True)
                    for o in p_outs[j]:
                        host_out[:o.numel()].view(o.shape).copy_(o, non_blocking=True)
                ev_out[ci].record(s_out)
        started[0] = True
    step()
    torch.cuda.synchronize()
    steps = max(1, args.e2e_steps)
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        step()
    torch.cuda.synchronize()
    dt = max_over_ranks(time.perf_counter() - t0, world)
    n_total = sum(sp.numel for sp in specs)
    return {"value": round(world * 2.0 * n_total * steps / dt / 1e9, 2), "unit": "GB/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": steps, "s_per_step": round(dt / steps, 4)}


# ---------------------------------------------------------------------------
# CPU oracle: baseline leg and the --impl reference arm
# ---------------------------------------------------------------------------
ORACLE_WEIGHTS_PER_CORE_S = 2.0e7   # about what one host core's oracle does per second (sizes the sample)


def oracle_pool_sample(samples, target_core_s: float, pool, region=None) -> dict:
    """Times the oracle as it stands (quantize, then reconstruct at k =
    1..4) on the host's cores.  Sampled matrices are taken in order until
    they hold about `target_core_s` core-seconds of oracle work (at least
    one), copied into shared memory (not timed), cut into about 4 row-range
    tasks per process, and timed from the first submission to the last
    result.  samples: (label, bf16 tensor) pairs."""
    from oracle.pool import Layout, SharedRegion, Task
    chosen, weights = [], 0
    for label, W in samples:
        chosen.append((label, W))
        weights += W.numel()
        if weights >= target_core_s * ORACLE_WEIGHTS_PER_CORE_S:
            break
    lay = Layout()
    offs = [lay.take(2 * W.numel()) for _, W in chosen]
    own = region is None
    reg = SharedRegion(lay.size) if own else region
    try:
        for (label, W), off in zip(chosen, offs):
            reg.array(off, np.uint16, W.numel())[:] = W.contiguous().view(torch.int16).cpu().numpy().view(
                np.uint16).reshape(-1)
        per_task = max(1 << 16, weights // (4 * pool.processes))
        tasks = []
        for (label, W), off in zip(chosen, offs):
            rows, cols = W.shape
            tasks += Task(reg.name, label, "asym", GROUP, STAGES, rows, cols, off, check=False,
                          oracle_prefixes=len(KS)).split(per_task)
        t0 = time.perf_counter()
        res = pool.run(tasks)
        wall = time.perf_counter() - t0
    finally:
        if own:
            reg.close()
    core_s = sum(r["seconds"] for r in res)
    names = [f"{label} {W.shape[0]}x{W.shape[1]}" for label, W in chosen]
    return {"bytes": 2.0 * weights, "weights": weights, "wall_s": wall, "core_s": core_s, "names": names}


def cpu_baseline(samples, target_core_s: float) -> dict:
    from oracle.pool import OraclePool, host_description
    host = host_description()
    with OraclePool() as pool:
        r = oracle_pool_sample(samples, target_core_s, pool)
        procs = pool.processes
    return {"value": round(r["bytes"] / r["wall_s"] / 1e9, 5), "unit": "GB/s", "cores": procs, "kind": "oracle",
            "sample": f"the single-threaded C oracle, quantize + reconstruct k=1..4, in {procs} processes over "
                      f"row ranges of {', '.join(r['names'])} ({r['weights']} weights, {r['wall_s']:.1f} s wall, "
                      f"{r['core_s']:.1f} core-s)",
            "per_core_gbs": round(r["bytes"] / r["core_s"] / 1e9, 5),
            "weights_per_s_per_core": round(r["weights"] / r["core_s"], 1),
            "cpu_model": host["cpu_model"], "host_cpus": host["cores"]}


REFERENCE_SAMPLE = ("q_proj", "k_proj", "v_proj", "o_proj")   # of layer 0, per step


def run_reference(args, world, rank):
    if rank != 0:
        return None
    from oracle.pool import OraclePool, host_description
    from paper_2608_04048_gb300 import workloads
    specs = [sp for sp in workloads.config_matrices(WORKLOAD)[:7] if sp.name.split(".")[-1] in REFERENCE_SAMPLE]
    samples = [(sp.name, workloads.generate(sp.rows, sp.cols, sp.seed, sp.dist, "cpu")) for sp in specs]
    host = host_description()
    with OraclePool() as pool:
        for _ in range(args.warmup):
            oracle_pool_sample(samples, float("inf"), pool)
        total_b, total_s, core_s = 0.0, 0.0, 0.0
        for _ in range(args.steps):
            r = oracle_pool_sample(samples, float("inf"), pool)
            total_b += r["bytes"]
            total_s += r["wall_s"]
            core_s += r["core_s"]
        procs = pool.processes
    value = total_b / total_s / 1e9
    names = ", ".join(f"{sp.name} {sp.rows}x{sp.cols}" for sp in specs)
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 5),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(total_s / max(1, args.steps) * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}: bounded sample of the same stack, {names}",
                   "step": f"oracle quantize + reconstruct k=1..4 of the sampled matrices on {procs} host "
                           f"processes (row ranges)"},
        "cpu_baseline": {"value": round(value, 5), "unit": "GB/s", "cores": procs, "kind": "oracle",
                         "sample": f"{names} per step", "per_core_gbs": round(total_b / core_s / 1e9, 5),
                         "cpu_model": host["cpu_model"]},
        "e2e": {"value": round(value, 5), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default=WORKLOAD,
                    help="single_4096, qwen3_8b_layer, qwen3_8b_stack (default), sweep_8192, qwen3_32b_stack")
    ap.add_argument("--split", action="store_true",
                    help="under torchrun: split ONE stack's matrices over the ranks (strong scaling)")
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-sym", action="store_true",
                    help="skip the symmetric binary16, base-checkpoint and product breakdown")
    ap.add_argument("--cpu-seconds", type=float, default=20.0,
                    help="core-seconds of oracle work in the CPU baseline (0 skips it)")
    ap.add_argument("--traffic-from", default=None,
                    help="write profiles/traffic.json from this ncu CSV of a qwen3_8b_layer run, and exit")
    ap.add_argument("--gemv-batches", default="1",
                    help="comma-separated activation-row counts for the decode-product breakdown (1..8)")
    args = ap.parse_args(argv)
    if args.traffic_from:
        record_traffic(args.traffic_from)
        return

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    try:
        if args.impl == "reference":
            line = run_reference(args, world, rank)
        else:
            if not torch.cuda.is_available():
                raise SystemExit("bench.py needs a CUDA device (use --impl reference for the CPU oracle)")
            line = run_gpu(args, world, rank, local)
        if line is not None:
            print(json.dumps(line), flush=True)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
