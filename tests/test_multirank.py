"""Multi-process paths on the CPU with the gloo backend (world size 2).

The hot path shards without any data exchange: under torchrun every rank
builds and processes its own independent stack, and the only collectives are
the timing barrier and the max-over-ranks of the elapsed time.  These tests
run that host logic with two gloo ranks, and the benchmark's reference arm
under torchrun (rank 0 prints one line, rank 1 exits cleanly)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, l = bench.dist_env()
        bench.barrier(w)
        mx = bench.max_over_ranks(float(10 + rank), w)
        q.put((rank, w, r, l, mx, bench.shard_seed_offset(rank)))
    finally:
        dist.destroy_process_group()


def test_gloo_two_ranks_max_and_shards():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    assert [x[0] for x in res] == [0, 1]
    assert all(x[1] == 2 for x in res)
    assert all(x[4] == 11.0 for x in res)           # max over ranks seen by every rank
    offsets = [x[5] for x in res]
    assert offsets[0] == 0 and offsets[1] > 10_000  # disjoint seeds: independent stacks


def test_reference_arm_under_torchrun_two_ranks():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
           "--steps", "1", "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle"


def _shard_worker(rank, world, port, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_04048_gb300 import workloads
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out = {}
        for name in ("qwen3_8b_stack", "qwen3_32b_stack", "qwen3_8b_layer"):
            specs = workloads.config_matrices(name)
            mine = bench.shard_matrices(specs, world, rank)
            got = [None] * world
            dist.all_gather_object(got, mine)
            out[name] = got
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_split_stack_covers_every_matrix_once(world):
    """--split: each rank computes its own share of ONE stack; gathered over
    gloo ranks, the shares cover every matrix exactly once and balance the
    weights to within one matrix."""
    from paper_2608_04048_gb300 import workloads
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    res = dict(q.get(timeout=10) for _ in range(world))
    for name, shares in res[0].items():
        assert all(res[r][name] == shares for r in range(world))  # every rank computes the same split
        specs = workloads.config_matrices(name)
        flat = sorted(i for s in shares for i in s)
        assert flat == list(range(len(specs))), name
        load = [sum(specs[i].numel for i in s) for s in shares]
        assert max(load) - min(load) <= max(sp.numel for sp in specs), (name, load)
