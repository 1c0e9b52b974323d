"""The N > 1 harness on CPU with gloo: ranks run independent batches (weak
scaling, no data-path collective); only the timing reduction crosses ranks."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        out[rank] = bench.max_over_ranks(1.5 + rank, True, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_with_gloo():
    world = 2
    # the manager's server process is spawned too: forking a process whose
    # earlier tests started torch's CPU threads can deadlock the child
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    assert dict(out) == {0: 2.5, 1: 2.5}


def test_ranks_draw_distinct_batches():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2606_01774_gb300 import workloads

    spec = workloads.WORKLOADS["tiny_fp32"]
    a = workloads.generate(spec.replace(seed=spec.seed + bench.rank_seed_offset(0)), linear=False)
    b = workloads.generate(spec.replace(seed=spec.seed + bench.rank_seed_offset(1)), linear=False)
    assert not torch.equal(a.softmax[0].q, b.softmax[0].q)


def test_reference_arm_under_torchrun_prints_once():
    """--impl reference under torchrun: rank 0 alone runs the CPU oracle and
    prints one JSON line; the other rank exits 0 without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0",
           "--workload", "tiny_fp32"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["n_gpus"] == 2
    assert d["cpu_baseline"]["kind"] == "oracle"
