"""Multi-rank plumbing of bench.py on CPU (gloo, world size 2).

Every rank quantizes its own layer (weak scaling, no data-path collective); the bench
only needs a barrier, a max over ranks of the step time, and rank-0-only output.  These
run here with gloo ranks; the GPU arm uses the same code with NCCL.
"""
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


def free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist(world)
    d.barrier()
    out[rank] = d.max(float(rank + 1) * 1.5)
    d.barrier()
    d.close()


def test_dist_barrier_and_max_over_ranks():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(world, free_port(), out), nprocs=world, join=True)
    assert out[0] == out[1] == 3.0


def _rank_leaves(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank), HSCALE_PG_TIMEOUT_S="5")
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist(world)
    d.barrier()
    if rank == 1:
        out[1] = "left"
        os._exit(0)                  # leaves between steps, with nothing in flight
    try:
        d.max(1.0)                   # the next collective of the surviving rank
        out[0] = "no error"
    except Exception as e:           # noqa: BLE001 -- any error is the expected outcome
        out[0] = type(e).__name__
    os._exit(0)


def test_a_rank_that_leaves_makes_the_next_collective_fail_not_hang():
    """Failure detection on the host: rank 1 exits between steps; rank 0's next
    collective must end with an error within the process-group timeout."""
    world = 2
    out = mp.Manager().dict()
    ctx = mp.start_processes(_rank_leaves, args=(world, free_port(), out), nprocs=world, join=False,
                             start_method="spawn")
    for _ in range(120):
        if ctx.join(timeout=1):       # True once every process has been joined
            break
    assert out.get(1) == "left"
    assert out.get(0) not in (None, "no error"), out.get(0)


def test_rank_layers_are_independent_problems():
    sys.path.insert(0, ROOT)
    from paper_2608_28113_gb300 import workloads as wl
    W = wl.WORKLOADS["layer-512x1024"]
    a = wl.weight(64, 64, W.sigma_w, W.seed + 7919 * 0)
    b = wl.weight(64, 64, W.sigma_w, W.seed + 7919 * 1)
    assert not torch.equal(a, b)
    assert torch.equal(a, wl.weight(64, 64, W.sigma_w, W.seed))   # reproducible per rank


def test_reference_arm_prints_once_under_torchrun():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes", "1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0",
           "--workload", "layer-512x1024"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["n_gpus"] == 2
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
