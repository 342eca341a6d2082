"""The profit experiment of Section 5.2 against Table 1, and the Section 5
post-processing helpers.

FCFS and LJF must reproduce Table 1 within the sampling noise of a
five-replication mean (the paper averages five replications); this pins the
workload recipe, the cost decomposition (Theorem "Profit decomposition") and
both baselines to numbers the paper prints.  ISJL does not reproduce its
Table 1 rows under the simulator's reading of Algorithm 2 (it is slower than LJF
on this workload, the table has it faster): the oracle's values are pinned in
tests/golden/profit_isjl_oracle.txt and the gap is asserted, as a finding.
"""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))
import make_profit_findings as F  # noqa: E402

from paper_2608_02244_gb300 import analysis  # noqa: E402

INF = 2**31 - 1
COLS = ("profit", "cost", "tau_Q", "c_T", "tau_E", "throughput", "avg_extent")


def _read(path):
    out = {}
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        pol, d, *vals = line.split()
        out[(pol, int(d))] = [float(v) for v in vals]
    return out


PAPER = _read(os.path.join(HERE, "golden", "table1_profit.txt"))
ORACLE = _read(os.path.join(HERE, "golden", "profit_isjl_oracle.txt"))


@pytest.fixture(scope="module")
def computed():
    return F.compute()


def test_fcfs_and_ljf_reproduce_table1(computed):
    recs, table = computed
    for key in [("fcfs", 0), ("ljf", 0)]:
        rec = recs[key]
        per_rep = {c: (analysis.avg_extent(rec) if c == "avg_extent" else np.asarray(rec[c], float)) for c in COLS}
        for j, c in enumerate(COLS):
            mean = per_rep[c].mean()
            sd5 = per_rep[c].std() / np.sqrt(5)          # noise of a five-replication mean
            assert abs(mean - PAPER[key][j]) <= 3 * sd5 + 1e-9, (key, c, mean, PAPER[key][j], sd5)


def test_ljf_has_zero_externality_and_extent(computed):
    recs, _ = computed
    assert (recs[("ljf", 0)]["E"] == 0).all() and (recs[("ljf", 0)]["max_extent"] == 0).all()


def test_isjl_oracle_values_pinned(computed):
    _, table = computed
    for key, vals in ORACLE.items():
        got = [table[key][c] for c in COLS] + [table[key]["T_make"]]
        np.testing.assert_allclose(got, vals, rtol=1e-9)


def test_isjl_table1_gap_is_a_finding(computed):
    """Table 1's ISJL throughput exceeds the oracle's by far more than the noise."""
    recs, table = computed
    for key, vals in PAPER.items():
        if key[0] != "isjl":
            continue
        thr = np.asarray(recs[key]["throughput"], float)
        sd5 = thr.std() / np.sqrt(5)
        assert vals[5] - thr.mean() > 3 * sd5, key
        # and the fairness budget still holds on every step of every replication
        assert (recs[key]["violations"] == 0).all()


def test_break_even_and_alpha_helpers(computed):
    recs, table = computed
    # Table 2's break-even needs ISJL to be faster than LJF; here it is not
    for a in (50, 100, 500):
        key = ("isjl", a)
        assert analysis.break_even_c(table[key]["tau_E"], table[("ljf", 0)]["T_make"], table[key]["T_make"]) is None
    assert analysis.break_even_c(1.35, 1000.0, 916.8) == pytest.approx(1.35 / 83.2)
    # alpha_cost: an ISJL run at alpha <= delta Q / O has E <= delta Q (E <= alpha O, Theorem 5)
    a, p, o, cnt = F.W.generate(6, 20, with_counts=True)
    from oracle import oracle as O
    for frac in (0.002, 0.01, 0.05):
        r0, _, _ = O.run("fcfs", 50, 0, INF, a, p, o, per_request=False, counts=cnt)
        for i in range(len(cnt)):
            alpha = int(analysis.alpha_cost(frac, r0["Q"][i], r0["O"][i]))
            ri, _, _ = O.run("isjl", 50, alpha, INF, a[i:i + 1], p[i:i + 1], o[i:i + 1], per_request=False,
                             counts=cnt[i:i + 1])
            assert ri["E"][0] <= frac * ri["Q"][0]
    # calibration: argmin c T + tau E, throughput floor, ties to the smaller alpha
    alphas = [50, 100, 150]
    assert analysis.calibrate_alpha(alphas, [1.0, 0.5, 0.5], [0.1, 0.2, 0.2]) == 100
    assert analysis.calibrate_alpha(alphas, [1.0, 0.5, 0.2], [0.1, 0.2, 0.2], [40, 41, 39], 40.5) == 100
    assert analysis.calibrate_alpha(alphas, [1.0, 0.5, 0.2], [0.1, 0.2, 0.2], [40, 41, 39], 45) is None
