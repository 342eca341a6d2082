"""GPU (C ABI, CUDA kernels) against the CPU oracle, record by record.

Integers (every counter and every per-request start / completion step) must
be bit-exact; the fp64 cost fields within 1e-12 relative (they are computed
from identical integers in the same order, so in practice they agree
exactly).  Both kernel variants (per-step and event-driven) are checked.
"""
import numpy as np
import pytest

from conftest import cuda_available

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

INF = 2**31 - 1
RTOL = 1e-12
F64 = ("c_T", "tau_Q", "tau_E", "cost", "revenue", "profit", "throughput", "ael")


@pytest.fixture(scope="module")
def S():
    from paper_2608_02244_gb300 import sim
    sim.lib()
    return sim


@pytest.fixture(scope="module")
def O(oracle_mod):
    return oracle_mod


def assert_records_equal(g, r, ctx=""):
    """g: GPU records, r: oracle records (same shape, structured)."""
    for f in r.dtype.names:
        if f in F64:
            np.testing.assert_allclose(g[f], r[f], rtol=RTOL, atol=0, err_msg=f"{ctx} {f}")
        else:
            np.testing.assert_array_equal(g[f], r[f], err_msg=f"{ctx} {f}")


def run_both(S, O, a, p, o, B, policies, deltas, kv, epoch, per_request=True, max_steps=0, check=True,
             counts=None, slack=None):
    n_inst, n = a.shape
    sm = S.Simulator(n_inst, n, B, max_steps=max_steps, epoch=epoch)
    try:
        res = sm.sweep(a, p, o, policies, deltas, kv, per_request=per_request, counts=counts, slack=slack)
    finally:
        sm.close()
    assert res["launches"] == 4
    assert (res["records"]["status"] != S.ISJL_ERR_INTERNAL).all()   # no kernel invariant ever fails
    if check:
        for i, (pol, d) in enumerate(zip(policies, deltas)):
            rec, st, co = O.run(pol, B, d, kv, a, p, o, max_steps=max_steps, per_request=per_request,
                                counts=counts, slack=slack)
            assert_records_equal(res["records"][i], rec, f"{pol} d={d} epoch={epoch}")
            if per_request:
                np.testing.assert_array_equal(res["start"][i], st, err_msg=f"start {pol} {d}")
                np.testing.assert_array_equal(res["completion"][i], co, err_msg=f"completion {pol} {d}")
    return res


EPOCHS = [False, True]


@pytest.mark.parametrize("epoch", EPOCHS)
def test_single_instance_workload(S, O, epoch):
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(1)
    run_both(S, O, a, p, o, 32, ["fcfs", "ljf", "isjl", "isjl", "isjl"], [32, 32, 32, 0, INF], 2048, epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
@pytest.mark.parametrize("B", [2, 3])
@pytest.mark.parametrize("kv", [16, INF])
def test_tiny_exhaustive_workload(S, O, epoch, B, kv):
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(2)
    pols = ["isjl"] * 5 + ["fcfs", "ljf", "sjf"] + ["isjl_beta"] * 3
    ds = [0, 1, 2, 4, INF, 0, 0, 0, 1, 2, 4]
    run_both(S, O, a, p, o, B, pols, ds, kv, epoch)


def test_tiny_exhaustive_competitive_ratio_on_gpu(S, O):
    """GPU makespans against the exhaustive optimum: B=2 meets 3/4 and CR(gamma)
    everywhere; B=3 misses exactly on the recorded instances."""
    import os
    import sys
    sys.path.insert(0, os.path.join(os.path.dirname(__file__), "golden"))
    import make_cr_findings as F
    from test_competitive_ratio import load_findings
    from paper_2608_02244_gb300 import workloads as W
    a, p, out = W.generate(2)
    o = p + out
    rec = load_findings()
    for B in (2, 3):
        sm = S.Simulator(len(a), 6, B, epoch=True)
        try:
            res = sm.sweep(a, p, out, ["isjl"] * 5, list(F.DELTAS), INF)
        finally:
            sm.close()
        for r, d in enumerate(F.DELTAS):
            T = res["records"][r]["T_make"]
            f34, fg = [], []
            for i in range(len(o)):
                topt = O.opt_makespan(a[i], o[i], B, d)
                m34, mg = F.misses(topt, int(T[i]), int(o[i].max()), d)
                if m34:
                    f34.append(i)
                if mg:
                    fg.append(i)
            if B == 2:
                assert f34 == [] and fg == []
            else:
                assert f34 == rec[(3, d, "3/4")] and fg == rec[(3, d, "gamma")]


@pytest.mark.parametrize("epoch", EPOCHS)
def test_online_sweep_workload_subset(S, O, epoch):
    """16 full-size instances (n = 1000, ragged against 32) of the online sweep."""
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(3, 16)
    pols = ["fcfs", "ljf"] + ["isjl"] * 5 + ["sjf", "isjl_beta", "isjl_beta"]
    ds = [0, 0, 16, 64, 256, 1024, INF, 0, 64, 1024]
    run_both(S, O, a, p, o, 256, pols, ds, 200_000, epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_heavy_tail_workload_subset(S, O, epoch):
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(4, 48)
    pols = ["fcfs", "ljf", "isjl", "isjl", "isjl", "sjf", "isjl_beta"]
    ds = [0, 0, 32, 128, 512, 0, 128]
    run_both(S, O, a, p, o, 128, pols, ds, 65_536, epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_large_instance_sample(S, O, epoch):
    """One instance of n = 100,000 (radix-sort path, two-level pending set)."""
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(5, [7])
    run_both(S, O, a, p, o, 512, ["fcfs", "ljf", "isjl"], [256, 256, 256], 1_000_000, epoch)


def test_online_sweep_full_size_sampled(S, O):
    """The benchmark's launch: all 10,000 instances x 7 runs in one sweep;
    sampled instances against the oracle, invariants on every record."""
    from paper_2608_02244_gb300 import workloads as W
    wl = W.WORKLOADS[3]
    a, p, o = W.generate(3)
    pols = ["fcfs", "ljf"] + ["isjl"] * 5
    ds = [0, 0, 16, 64, 256, 1024, INF]
    for epoch in EPOCHS:
        sm = S.Simulator(wl.n_instances, wl.n_per_instance, 256, epoch=epoch)
        try:
            res = sm.sweep(a, p, o, pols, ds, 200_000, per_request=True)
        finally:
            sm.close()
        assert res["status"] == 0
        R = res["records"]
        assert (R["status"] == 0).all()
        assert (R["W"] == R["Q"] + R["E"]).all() and (R["token_adv"] == R["O"]).all()
        assert (R["violations"][1:] == 0).all() and (R["kv_violations"] == 0).all()
        assert (R["peak_kv"] <= 200_000).all() and (R["peak_batch"] <= 256).all()
        sample = [0, 1, 977, 2048, 4099, 5555, 8191, 9999]
        for i, (pol, d) in enumerate(zip(pols, ds)):
            rec, st, co = O.run(pol, 256, d, 200_000, a[sample], p[sample], o[sample])
            assert_records_equal(R[i][sample], rec, f"full {pol} {d} epoch={epoch}")
            np.testing.assert_array_equal(res["start"][i][sample], st)
            np.testing.assert_array_equal(res["completion"][i][sample], co)
            # summaries: exact integer totals, fp64 within tolerance
            s = res["summaries"][i]
            assert s["T_busy"] == int(R[i]["T_busy"].sum()) and s["E"] == int(R[i]["E"].sum())
            assert s["n_ok"] == wl.n_instances and s["status"] == 0
            np.testing.assert_allclose(s["cost"], R[i]["cost"].sum(), rtol=1e-12)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_profit_experiment_workload_ragged(S, O, epoch):
    """Section 5.2's design: instances of 150-250 accepted requests in 400 slots."""
    from paper_2608_02244_gb300 import workloads as W
    a, p, o, cnt = W.generate(6, 64, with_counts=True)
    assert cnt.min() < 400
    pols = ["fcfs", "ljf"] + ["isjl"] * 7 + ["sjf", "isjl_beta"]
    ds = [0, 0, 50, 100, 150, 250, 300, 400, 500, 0, 150]
    run_both(S, O, a, p, o, 50, pols, ds, INF, epoch, counts=cnt)


@pytest.mark.parametrize("epoch", EPOCHS)
@pytest.mark.parametrize("B", [2, 3])
def test_tiny_robust_workload(S, O, epoch, B):
    """Robust-ISJL: plans with u = o + slack, serves o (Section 3.3)."""
    from paper_2608_02244_gb300 import workloads as W
    a, p, o, e = W.generate(7, with_slack=True)
    pols = ["isjl"] * 5 + ["fcfs", "ljf", "sjf", "isjl_beta"]
    ds = [0, 1, 2, 4, INF, 0, 0, 0, 2]
    for kv in (16, INF):
        run_both(S, O, a, p, o, B, pols, ds, kv, epoch, slack=e)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_online_robust_workload_subset(S, O, epoch):
    from paper_2608_02244_gb300 import workloads as W
    a, p, o, e = W.generate(8, 12, with_slack=True)
    pols = ["fcfs", "ljf", "isjl", "isjl", "isjl", "sjf", "isjl_beta"]
    ds = [0, 0, 16, 256, INF, 0, 256]
    run_both(S, O, a, p, o, 256, pols, ds, 200_000, epoch, slack=e)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_ragged_counts_edges(S, O, epoch):
    """Empty instances, full instances, and an out-of-range count (INVALID_ARG)."""
    rng = np.random.default_rng(9)
    n = 70
    a = np.sort(rng.integers(0, 90, (6, n)), axis=1).astype(np.int32)
    p = rng.integers(0, 20, (6, n)).astype(np.int32)
    o = rng.integers(1, 60, (6, n)).astype(np.int32)
    cnt = np.array([0, n, 1, 33, 0, 64], np.int32)
    run_both(S, O, a, p, o, 8, ["fcfs", "ljf", "isjl", "isjl", "sjf", "isjl_beta"], [0, 0, 4, INF, 0, 4], 200, epoch,
             counts=cnt)
    e = rng.integers(0, 15, (6, n)).astype(np.int32)        # with predictions as well
    run_both(S, O, a, p, o, 8, ["fcfs", "ljf", "isjl", "isjl", "sjf", "isjl_beta"], [0, 0, 4, INF, 0, 4], 300, epoch,
             counts=cnt, slack=e)
    bad = cnt.copy()
    bad[2] = n + 1
    res = run_both(S, O, a, p, o, 8, ["isjl"], [4], 200, epoch, counts=bad, check=False)
    assert res["records"][0]["status"][2] == 1 and (np.delete(res["records"][0]["status"], 2) == 0).all()
    rec, _, _ = O.run("isjl", 8, 4, 200, a, p, o, counts=bad)
    assert_records_equal(res["records"][0], rec)


# ---- edge cases -------------------------------------------------------------
def _inst(rows):
    a = np.array([r[0] for r in rows], np.int32)
    p = np.array([r[1] for r in rows], np.int32)
    o = np.array([r[2] for r in rows], np.int32)
    return a, p, o


@pytest.mark.parametrize("epoch", EPOCHS)
def test_edge_shapes(S, O, epoch):
    rng = np.random.default_rng(7)
    cases = []
    # n = 1; B = 1; n = 33 (two bitset words); B = 512 with few requests; idle gaps
    for n, B in [(1, 1), (1, 4), (33, 1), (33, 3), (64, 512), (200, 64), (97, 2)]:
        a = np.sort(rng.integers(0, 400, (5, n)), axis=1).astype(np.int32)
        p = rng.integers(0, 30, (5, n)).astype(np.int32)
        o = rng.integers(1, 90, (5, n)).astype(np.int32)
        cases.append((a, p, o, B))
    for a, p, o, B in cases:
        kv = int((p + o).max()) + 50
        run_both(S, O, a, p, o, B, ["fcfs", "ljf", "isjl", "isjl", "isjl", "sjf", "isjl_beta"],
                 [0, 0, 0, 5, INF, 0, 5], kv, epoch)
        run_both(S, O, a, p, o, B, ["isjl", "isjl", "sjf", "isjl_beta"], [3, 40, 0, 40], INF, epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_radix_path_small_count(S, O, epoch):
    """n = 4097 takes the radix sort; long idle gaps between arrivals."""
    rng = np.random.default_rng(8)
    n = 4097
    a = np.sort(rng.integers(0, 30000, (2, n)), axis=1).astype(np.int32)
    p = rng.integers(0, 200, (2, n)).astype(np.int32)
    o = rng.integers(1, 300, (2, n)).astype(np.int32)
    run_both(S, O, a, p, o, 40, ["fcfs", "ljf", "isjl", "isjl", "sjf", "isjl_beta"], [0, 0, 60, INF, 0, 60], 3000,
             epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_error_statuses(S, O, epoch):
    a = np.zeros((4, 3), np.int32)
    p = np.zeros((4, 3), np.int32)
    o = np.array([[3, 2, 1], [3, 0, 1], [3, 2, 1], [9, 2, 1]], np.int32)
    a[2] = [0, 2, 1]               # decreasing arrivals
    res = run_both(S, O, a, p, o, 2, ["fcfs", "isjl"], [0, 1], 8, epoch, check=False)
    R = res["records"]
    assert list(R["status"][0]) == [0, 2, 1, 2]   # ok, o=0 infeasible, invalid, o > kv infeasible
    assert res["status"] in (1, 2)
    for i, (pol, d) in enumerate([("fcfs", 0), ("isjl", 1)]):
        rec, _, _ = O.run(pol, 2, d, 8, a, p, o)
        np.testing.assert_array_equal(R[i]["status"], rec["status"])
        assert_records_equal(R[i][:1], rec[:1])
    # the step guard returns an error status instead of trapping
    res = run_both(S, O, a[:1], p[:1], o[:1], 2, ["isjl"], [0], 8, epoch, max_steps=2, check=False)
    assert res["records"][0]["status"][0] == 5 and res["status"] == 5


@pytest.mark.parametrize("epoch", EPOCHS)
def test_step_limit_partial_records(S, O, epoch):
    """A run stopped by max_steps reports exactly the steps 0..max_steps it
    served, like the oracle: counters, partial W and E, the requests finished
    by then, and -1 for requests that did not start or finish.  The guard is
    also put one step before and at a completion step (the retire boundary)."""
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(3, 4)
    pols = ["fcfs", "ljf", "isjl", "isjl", "sjf"]
    ds = [0, 0, 64, INF, 0]
    full, _, co = O.run("fcfs", 256, 0, 200_000, a[:1], p[:1], o[:1])
    c_mid = int(np.sort(co[0])[len(co[0]) // 2])
    for ms in (1, 37, 1500, c_mid - 1, c_mid):
        res = run_both(S, O, a, p, o, 256, pols, ds, 200_000, epoch, max_steps=ms)
        assert (res["records"][0]["status"] == 5).all() and res["status"] == 5
        assert (res["start"] == -1).any() and (res["completion"] == -1).any()


@pytest.mark.parametrize("epoch", EPOCHS)
def test_bulk_starts_with_ties_and_partial_rows(S, O, epoch):
    """Admissions that start many requests at once (the 32-wide bulk path):
    lengths from a tiny set (long runs of equal o, so SJF and LJF take large
    tie groups in index order), B spanning several register rows with a
    partial last row, every request at t = 0 or in bursts, with and without a
    KV cap that stops a bulk in its middle."""
    rng = np.random.default_rng(21)
    n = 300
    a = np.zeros((6, n), np.int32)
    a[3:] = np.sort(rng.integers(0, 40, (3, n)), axis=1)          # bursts of arrivals
    p = np.zeros((6, n), np.int32)
    o = rng.choice(np.array([3, 7, 7, 12, 40], np.int32), (6, n)).astype(np.int32)
    pols = ["fcfs", "ljf", "sjf", "isjl", "isjl", "isjl", "isjl_beta"]
    ds = [0, 0, 0, 4, 30, INF, 8]
    for B in (33, 100, 256):
        for kv in (INF, 700):
            run_both(S, O, a, p, o, B, pols, ds, kv, epoch)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_domain_limits(S, O, epoch):
    """The GPU's documented limits, against the oracle just below them: a
    request of ISJL_MAX_LEN = 65,535 tokens, and an instance whose
    sum o + max arrival is 2^30 - 2 (the step counter's range), run and agree
    with the oracle; one token more at either limit is INVALID_ARG on the GPU
    (the oracle has no such limit and simulates it)."""
    # o_i = 65,535 next to short requests, with arrivals
    a = np.array([[0, 0, 3, 9]], np.int32)
    p = np.array([[65000, 3, 0, 7]], np.int32)
    o = np.array([[535, 4, 11, 2]], np.int32)
    run_both(S, O, a, p, o, 2, ["fcfs", "ljf", "isjl", "sjf"], [0, 0, 6, 0], INF, epoch)
    o2 = o.copy()
    o2[0, 0] += 1                                   # 65,536 tokens
    res = run_both(S, O, a, p, o2, 2, ["fcfs"], [0], INF, epoch, check=False)
    assert res["records"][0]["status"][0] == S.ISJL_ERR_INVALID_ARG
    # sum o + max arrival = 2^30 - 2: 16,384 requests of 65,535 tokens and one of 16,382
    n = 16_385
    a = np.zeros((1, n), np.int32)
    p = np.full((1, n), 65_000, np.int32)
    o = np.full((1, n), 535, np.int32)
    p[0, -1] = 0                                    # the last request: 16,382 tokens in all
    o[0, -1] = 16_382
    assert int((p + o).astype(np.int64).sum()) == 2**30 - 2
    run_both(S, O, a, p, o, 512, ["fcfs", "ljf"], [0, 0], INF, epoch, per_request=False)
    o3 = o.copy()
    o3[0, -1] += 1                                  # sum o + max arrival = 2^30 - 1
    res = run_both(S, O, a, p, o3, 512, ["fcfs"], [0], INF, epoch, per_request=False, check=False)
    assert res["records"][0]["status"][0] == S.ISJL_ERR_INVALID_ARG


def test_integer_rate_probe(S):
    """The roofline denominators: both probe kinds run, count their
    instructions and report a rate within what 152 SMs can issue."""
    import torch
    for kind in (0, 1):
        n, ms = S.isjl_probe_int_rate(kind, 200)
        props = torch.cuda.get_device_properties(0)
        blocks = n / (256 * 200 * 128)          # one full wave: a whole number of blocks per SM
        assert blocks == int(blocks) and int(blocks) % props.multi_processor_count == 0
        rate = n / (ms / 1e3)
        # at most 128 lanes per SM at 2.2 GHz, and surely more than 1 Tops/s
        assert 1e12 < rate < props.multi_processor_count * 128 * 2.2e9, (kind, rate)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_completion_windows(S, O, epoch):
    """Instances where the event-driven kernel serves long completion windows:
    bursts of arrivals (many requests start at the same step), lengths from a
    small set (ties in completion and in start), LJF batches and ISJL with a
    gate shut for most of a stage (alpha 0, 2, 8, 64), with and without a KV
    cap, and step guards that stop a run inside a window."""
    rng = np.random.default_rng(33)
    n = 300
    a = np.sort(rng.choice(np.array([0, 0, 0, 40, 120, 121, 500], np.int32), (4, n)), axis=1).astype(np.int32)
    p = rng.integers(0, 3, (4, n)).astype(np.int32)
    o = rng.choice(np.array([1, 5, 5, 9, 30, 31, 200], np.int32), (4, n)).astype(np.int32)
    pols = ["ljf", "isjl", "isjl", "isjl", "isjl", "isjl_beta", "fcfs"]
    ds = [0, 0, 2, 8, 64, 8, 0]
    for B in (8, 64):
        for kv in (INF, 900):
            run_both(S, O, a, p, o, B, pols, ds, kv, epoch)
        for ms in (37, 401, 1500):
            run_both(S, O, a, p, o, B, pols, ds, 900, epoch, max_steps=ms)


@pytest.mark.parametrize("epoch", EPOCHS)
def test_random_configurations(S, O, epoch):
    """Randomised shapes against the oracle, every policy: request counts
    from 1 to 300 (ragged counts on some), B from 1 to 512 (every register
    row count), budgets from 0 to infinity, KV caps from the largest request
    upwards or none, arrivals offline, spread or in bursts, lengths with many
    ties or spread out, upper-bound slack on some, step guards on some."""
    rng = np.random.default_rng(2024)
    pols = ["fcfs", "ljf", "sjf", "isjl", "isjl", "isjl", "isjl_beta"]
    for case in range(60):
        n_inst = int(rng.integers(1, 5))
        n = int(rng.choice([1, 2, 7, 33, 64, 150, 300]))
        B = int(rng.choice([1, 2, 3, 31, 32, 33, 64, 100, 128, 129, 256, 257, 384, 512]))
        kind = case % 3
        if kind == 0:
            a = np.zeros((n_inst, n), np.int32)
        elif kind == 1:
            a = np.sort(rng.integers(0, 5 * n + 1, (n_inst, n)), axis=1).astype(np.int32)
        else:
            a = np.sort(rng.choice(np.array([0, 3, 3, 50, 51, 400]), (n_inst, n)), axis=1).astype(np.int32)
        if case % 2:
            o = rng.choice(np.array([1, 4, 4, 9, 16, 16, 70]), (n_inst, n)).astype(np.int32)
        else:
            o = rng.integers(1, 400, (n_inst, n)).astype(np.int32)
        p = rng.integers(0, 3, (n_inst, n)).astype(np.int32)      # o_i = prompt + output >= 1
        o = np.where(p + np.maximum(o - p, 0) < 1, 1, np.maximum(o - p, 0)).astype(np.int32)
        big = int((p + o).max())
        e = rng.integers(0, 20, (n_inst, n)).astype(np.int32) if case % 4 == 3 else None
        big_u = big + (int(e.max()) if e is not None else 0)
        kv = INF if case % 5 == 0 else int(rng.integers(big_u, big_u * 6 + 2))
        ds = [0, 0, 0, 0, int(rng.integers(1, 40)), INF, int(rng.integers(1, 40))]
        counts = rng.integers(0, n + 1, n_inst).astype(np.int32) if case % 6 == 5 else None
        ms = int(rng.integers(1, 3 * n + 5)) if case % 7 == 6 else 0
        run_both(S, O, a, p, o, B, pols, ds, kv, epoch, counts=counts, slack=e, max_steps=ms)


def test_invalid_arguments_rejected(S):
    import torch
    sm = S.Simulator(1, 4, 2)
    try:
        x = torch.zeros(4, dtype=torch.int32, device="cuda")
        rec, _, _ = sm.buffers(1, False)
        assert S.isjl_sim_run(sm.handle, 2, -1, 10, x, x, x, rec) == S.ISJL_ERR_INVALID_ARG
        assert S.isjl_sim_run(sm.handle, 2, 1, 0, x, x, x, rec) == S.ISJL_ERR_INVALID_ARG
        assert S.isjl_sim_run(sm.handle, 7, 1, 10, x, x, x, rec) == S.ISJL_ERR_INVALID_ARG
    finally:
        sm.close()
    with pytest.raises(S.IsjlError):
        S.isjl_sim_create(1, 4, 513)
    with pytest.raises(S.IsjlError):
        S.isjl_sim_create(0, 4, 2)


def test_sweep_equals_single_runs_and_host_entry_point(S, O):
    import torch
    from paper_2608_02244_gb300 import workloads as W
    a, p, o = W.generate(3, 8)
    pols, ds = ["fcfs", "isjl", "isjl"], [0, 64, INF]
    sm = S.Simulator(8, 1000, 256, epoch=True)
    try:
        res = sm.sweep(a, p, o, pols, ds, 200_000)
        for i, (pol, d) in enumerate(zip(pols, ds)):
            one = sm.sweep(a, p, o, [pol], [d], 200_000)
            assert res["records"][i].tobytes() == one["records"][0].tobytes()
        pin = [torch.from_numpy(np.ascontiguousarray(x)).pin_memory() for x in (a, p, o)]
        hrec = torch.empty(len(pols) * 8 * S.RECORD_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
        st = S.isjl_sim_run_sweep_host(sm.handle, pols, ds, 200_000, *pin, hrec)
        assert st == 0
        host = hrec.numpy().view(S.RECORD_DTYPE).reshape(len(pols), 8)
        assert host.tobytes() == res["records"].tobytes()
    finally:
        sm.close()
    # with per-instance counts and upper-bound slack, through host memory
    a, p, o, cnt = W.generate(6, 16, with_counts=True)
    e = np.random.default_rng(3).integers(0, 50, a.shape).astype(np.int32)
    pols, ds = ["fcfs", "ljf", "isjl", "sjf"], [0, 0, 150, 0]
    sm = S.Simulator(16, 400, 50)
    try:
        res = sm.sweep(a, p, o, pols, ds, INF, counts=cnt, slack=e)
        pin = [torch.from_numpy(np.ascontiguousarray(x)).pin_memory() for x in (a, p, o, cnt, e)]
        hrec = torch.empty(len(pols) * 16 * S.RECORD_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
        st = S.isjl_sim_run_sweep_host(sm.handle, pols, ds, INF, *pin[:3], hrec, h_count=pin[3], h_slack=pin[4])
        assert st == 0
        host = hrec.numpy().view(S.RECORD_DTYPE).reshape(len(pols), 16)
        assert host.tobytes() == res["records"].tobytes()
        for i, (pol, d) in enumerate(zip(pols, ds)):
            rec, _, _ = O.run(pol, 50, d, INF, a, p, o, per_request=False, counts=cnt, slack=e)
            assert_records_equal(host[i], rec, f"host {pol}")
    finally:
        sm.close()
