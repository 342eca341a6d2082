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
  large instances (1,024 x 100,000, FCFS, LJF, ISJL): every instance's integer
      record fields and per-request start and completion steps against the
      oracle's stored per-instance digests (the oracle needs 10-30 s per
      instance, so tests/golden/make_large_digest.py ran it once on all of them),
      and 8 spread-out instances against the oracle run here, field by field.

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
    sample = np.linspace(0, 1023, 8).astype(int)
    check_workload(S, pool, 5, ["fcfs", "ljf", "isjl"], [0, 0, 256], per_request=True, sample=sample)


def _golden_digest_module():
    import importlib.util
    import os
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "make_large_digest.py")
    spec = importlib.util.spec_from_file_location("make_large_digest", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_large_instance_every_instance_digest(S, pool):
    """All 1,024 large instances, both kernels, against the oracle's digests.
    An instance whose generated inputs do not match the stored input digest
    (a platform whose floating-point draws differ) is checked against the
    oracle run here instead."""
    import os
    from oracle import parallel
    from paper_2608_02244_gb300 import workloads as W
    D = _golden_digest_module()
    stored = {}
    with open(os.path.join(os.path.dirname(D.__file__), "large_instance_digest.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            i, din, dres = line.split()
            stored[int(i)] = (din, dres)
    wl = W.WORKLOADS[D.WID]
    assert sorted(stored) == list(range(wl.n_instances))
    B, kv = wl.B[0], wl.kv_caps[0]
    pols, ds = [r[0] for r in D.RUNS], [r[1] for r in D.RUNS]
    a, p, o = W.generate(D.WID)
    same = np.array([D.input_digest(a[i], p[i], o[i]) == stored[i][0] for i in range(wl.n_instances)])
    redo = np.flatnonzero(~same)
    t = time.perf_counter()
    for ep in (False, True):
        res = gpu_sweep(S, a, p, o, B, pols, ds, kv, ep, per_request=True)
        rec, st, co = res["records"], res["start"], res["completion"]
        bad = [i for i in np.flatnonzero(same)
               if D.result_digest([rec[r][i] for r in range(len(pols))], [st[r][i] for r in range(len(pols))],
                                  [co[r][i] for r in range(len(pols))]) != stored[i][1]]
        assert not bad, f"epoch={ep}: {len(bad)} instances differ from the oracle, first {bad[:8]}"
        for r, (pol, d) in enumerate(zip(pols, ds)):
            if redo.size:
                orec, ost, oco = parallel.run(pool, pol, B, d, kv, a[redo], p[redo], o[redo], per_request=True)
                assert_records_equal(rec[r][redo], orec, f"w5 {pol} d={d} epoch={ep} (inputs drawn differently)")
                np.testing.assert_array_equal(st[r][redo], ost)
                np.testing.assert_array_equal(co[r][redo], oco)
        del res, rec, st, co
    print(f"large instances: {int(same.sum())} by digest, {redo.size} by the oracle here, "
          f"{time.perf_counter() - t:.0f} s")
