"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): each rank
simulates an independent replica of the workload, and the whole-job figures
are the max of the timings and the sum of the units over ranks."""
import os
import socket

import numpy as np
import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t, u, e = bench.combine_ranks(10.0 + rank, 100.0 * (rank + 1), 20.0 - rank, dist, "cpu")
    out[rank] = (t, u, e)
    dist.barrier()
    dist.destroy_process_group()


def test_combine_ranks_gloo_world2():
    import torch.multiprocessing as mp
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    for r in range(2):
        assert out[r] == (11.0, 300.0, 20.0)


def test_single_rank_passthrough():
    import bench
    assert bench.combine_ranks(5.0, 7.0, 9.0, None) == (5.0, 7.0, 9.0)


def test_rank_replicas_are_independent_instances():
    from paper_2608_02244_gb300 import workloads as W
    a0, p0, o0 = W.generate(3, 2, replica=0)
    a1, p1, o1 = W.generate(3, 2, replica=1)
    assert not np.array_equal(p0, p1) and a0.shape == a1.shape
    a0b, _, _ = W.generate(3, 2)
    np.testing.assert_array_equal(a0, a0b)


def test_reference_arm_prints_one_json_line():
    """bench.py --impl reference times the oracle on the host and prints one
    JSON line with the contract's keys (a small workload, one host process)."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload", "2",
                          "--oracle-cores", "1", "--steps", "1", "--warmup", "0"],
                         capture_output=True, text=True, timeout=300, check=True).stdout
    lines = [l for l in out.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]


def test_run_grids_are_valid():
    import bench
    from paper_2608_02244_gb300 import workloads as W
    for wid, (pols, deltas, per_core) in bench.GRIDS.items():
        assert wid in W.WORKLOADS and len(pols) == len(deltas) <= 32 and per_core >= 1
        assert set(pols) <= {"fcfs", "ljf", "isjl", "sjf", "isjl_beta"}


def test_epoch_count_counts_distinct_event_steps():
    """The event-driven kernel's algorithmic work counts epochs: per (run,
    instance), the distinct steps at which some request starts or completes;
    -1 entries (requests that never started or finished) are not steps."""
    import bench
    start = np.array([[[0, 0, 3, -1], [5, 5, 5, 5]]], np.int32)          # 1 run, 2 instances, n = 4
    compl = np.array([[[3, 4, 9, -1], [6, 7, 7, 8]]], np.int32)
    # instance 0: {0, 3, 4, 9} -> 4; instance 1: {5, 6, 7, 8} -> 4
    assert bench.epoch_count(start, compl) == 8
    two = np.concatenate([start, start])
    assert bench.epoch_count(two, np.concatenate([compl, compl])) == 16
    assert bench.epoch_count(np.full((1, 1, 3), -1, np.int32), np.full((1, 1, 3), -1, np.int32)) == 0
