"""bench.py's N>1 host logic on CPU with gloo, world size 2.

The data path has no exchange step: every rank runs its own replica of the
workload, and ranks only meet to time (barrier, max of elapsed times) and to
add up the work done.  These tests run that logic in two processes, and the
reference arm under torchrun, where rank 0 alone runs the oracle and prints.
"""
import json
import os
import socket
import subprocess
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    bench.barrier(ws)
    t = bench.max_over_ranks(10.0 + rank, ws, torch.device("cpu"))
    n = bench.sum_over_ranks(100.0 * (rank + 1), ws, torch.device("cpu"))
    out[rank] = (t, n)
    dist.destroy_process_group()


def test_timing_aggregation_over_two_ranks():
    ws = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(ws, free_port(), out), nprocs=ws, join=True)
        res = dict(out)
    # every rank sees the slowest rank's time and the work of all ranks
    assert res[0] == res[1] == (11.0, 300.0)


def test_reference_arm_under_torchrun_prints_once():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()), "bench.py", "--impl",
           "reference", "--workload", "tiny_mf", "--gpus", "2", "--steps", "3", "--warmup", "3",
           "--cpu-budget", "1"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"]["h2d_bytes_per_step"] == 0


def test_reference_arm_with_relocation_timing_and_versioned_refresh():
    # the placement, timing and refresh options reach the oracle the reference arm times
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny_mf", "--steps", "3",
           "--warmup", "3", "--cpu-budget", "1", "--relocate", "--timing", "adaptive", "--delta-refresh"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    d = json.loads([ln for ln in r.stdout.splitlines() if ln.startswith("{")][0])
    assert d["impl"] == "reference" and d["value"] > 0
    assert (d["config"]["placement"], d["config"]["action_timing"], d["config"]["refresh"]) == (
        "relocate", "adaptive", "versioned")
