"""Whole-workload parity: the benchmark's sweeps against the oracle, record by
record.

  online delta-sweep (10,000 instances x 1,000 requests, FCFS, LJF and ISJL at
      five budgets, plus SJF and Algorithm "ISJL" with beta): every record and
      every per-request start and completion;
  heavy-tail mix (100,000 x 500, FCFS, LJF, ISJL at three budgets): every record;
  online-robust (10,000 x 1,000 with upper-bound slack, the delta-sweep's runs):
      every record;
  profit experiment (10,000 ragged instances of up to 400, FCFS, LJF, ISJL at
      seven budgets): every record;
  large instances (1,024 x 100,000, FCFS, LJF, ISJL): the GPU simulates all of
      them; the oracle (about 30 s per instance) checks the records and
      per-request steps of 24 spread-out instances.

Both kernel variants run; the oracle runs once, on every host core (a spawned
process pool), and both are compared with it.  Integers bit-exact, fp64 within
1e-12 relative; no record may carry the internal-error status.
"""
import time

import numpy as np
import pytest

from conftest import cuda_available
from test_parity_gpu import F64, RTOL, assert_records_equal

pytestmark = [pytest.mark.gpu, pytest.mark.slow,
              pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

INF = 2**31 - 1
INTERNAL = 7


@pytest.fixture(scope="module")
def pool():
    from oracle import parallel
    p = parallel.make_pool()
    yield p
    p.close()
    p.join()


@pytest.fixture(scope="module")
def S():
    from paper_2608_02244_gb300 import sim
    sim.lib()
    return sim


def gpu_sweep(S, a, p, o, B, pols, ds, kv, epoch, per_request, counts=None, slack=None):
    sm = S.Simulator(len(a), a.shape[1], B, epoch=epoch)
    try:
        res = sm.sweep(a, p, o, pols, ds, kv, per_request=per_request, counts=counts, slack=slack)
    finally:
        sm.close()
    assert (res["records"]["status"] != INTERNAL).all()
    return res


def check_workload(S, pool, wid, pols, ds, per_request, sample=None):
    from oracle import parallel
    from paper_2608_02244_gb300 import workloads as W
    wl = W.WORKLOADS[wid]
    B, kv = wl.B[0], wl.kv_caps[0]
    a, p, o, cnt, e = W.generate(wid, with_counts=True, with_slack=True)
    cnt = cnt if wl.ragged else None
    e = e if wl.robust else None
    res = {ep: gpu_sweep(S, a, p, o, B, pols, ds, kv, ep, per_request, cnt, e) for ep in (False, True)}
    rows = np.arange(len(a)) if sample is None else np.asarray(sample)
    t = time.perf_counter()
    for i, (pol, d) in enumerate(zip(pols, ds)):
        rec, st, co = parallel.run(pool, pol, B, d, kv, a[rows], p[rows], o[rows], per_request=per_request,
                                   counts=None if cnt is None else cnt[rows], slack=None if e is None else e[rows])
        for ep, r in res.items():
            assert_records_equal(r["records"][i][rows], rec, f"w{wid} {pol} d={d} epoch={ep}")
            if per_request:
                np.testing.assert_array_equal(r["start"][i][rows], st, err_msg=f"w{wid} start {pol} {d} {ep}")
                np.testing.assert_array_equal(r["completion"][i][rows], co, err_msg=f"w{wid} compl {pol} {d} {ep}")
    print(f"workload {wid}: {len(rows)} instances x {len(pols)} runs checked, oracle {time.perf_counter() - t:.0f} s")


def test_online_delta_sweep_every_record(S, pool):
    check_workload(S, pool, 3, ["fcfs", "ljf"] + ["isjl"] * 5 + ["sjf", "isjl_beta"],
                   [0, 0, 16, 64, 256, 1024, INF, 0, 256], per_request=True)


def test_heavy_tail_every_record(S, pool):
    check_workload(S, pool, 4, ["fcfs", "ljf", "isjl", "isjl", "isjl"], [0, 0, 32, 128, 512], per_request=False)


def test_online_robust_every_record(S, pool):
    check_workload(S, pool, 8, ["fcfs", "ljf"] + ["isjl"] * 5, [0, 0, 16, 64, 256, 1024, INF], per_request=False)


def test_profit_experiment_every_record(S, pool):
    check_workload(S, pool, 6, ["fcfs", "ljf"] + ["isjl"] * 7, [0, 0, 50, 100, 150, 250, 300, 400, 500],
                   per_request=False)


def test_large_instance_spread_sample(S, pool):
    sample = np.linspace(0, 1023, 24).astype(int)
    check_workload(S, pool, 5, ["fcfs", "ljf", "isjl"], [0, 0, 256], per_request=True, sample=sample)
