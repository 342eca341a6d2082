"""The reading study of Algorithm 2 (tests/golden/isjl_reading_study.txt).

The study switches one open reading of the oracle's ISJL at a time and
records, for each, the Section 5.2 profit experiment and the tiny-exhaustive
competitive-ratio checks.  These tests re-derive part of the file, tie its
specification rows to the other pinned findings, and assert what the study
shows: no reading that keeps Eq. 1 on every step reaches Table 1's ISJL
throughput (or even LJF's, beyond noise), and the one that drops the gate on
plan entries breaks Eq. 1 without reaching Table 1 either.
"""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))
import make_reading_study as RS  # noqa: E402

from oracle import oracle as O  # noqa: E402

INF = 2**31 - 1


def _load():
    prof, tiny = {}, {}
    for line in open(os.path.join(HERE, "golden", "isjl_reading_study.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        if f[1] == "profit":
            prof[(f[0], int(f[2]))] = (float(f[3]), float(f[4]), float(f[5]), int(f[6]))
        else:
            tiny[(f[0], int(f[2]), int(f[3]))] = (int(f[4]), int(f[5]), float(f[6]), int(f[7]))
    return prof, tiny


PROF, TINY = _load()


def _table1_isjl_throughput():
    out = {}
    for line in open(os.path.join(HERE, "golden", "table1_profit.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        if f[0] == "isjl":
            out[int(f[1])] = float(f[7])
    return out


def test_variant_zero_is_the_specified_oracle():
    from paper_2608_02244_gb300 import workloads as W
    a, p, o, cnt = W.generate(6, 12, with_counts=True)
    for d in (50, 250):
        r0, s0, c0 = O.run("isjl", 50, d, INF, a, p, o, counts=cnt)
        r1, s1, c1 = O.run("isjl", 50, d, INF, a, p, o, counts=cnt, variant=0)
        assert r0.tobytes() == r1.tobytes()
        np.testing.assert_array_equal(s0, s1)
        np.testing.assert_array_equal(c0, c1)


def test_spec_rows_agree_with_the_pinned_findings():
    """The study's specification rows repeat the profit and CR findings."""
    import make_cr_findings as CR
    from test_competitive_ratio import load_findings
    rec = load_findings()
    for d in RS.TINY_DELTAS:
        m34, mg, _, viol = TINY[("spec", 3, d)]
        assert m34 == len(rec[(3, d, "3/4")]) and mg == len(rec[(3, d, "gamma")]) and viol == 0
        assert TINY[("spec", 2, d)][:2] == (0, 0)
    pinned = {}
    for line in open(os.path.join(HERE, "golden", "profit_isjl_oracle.txt")):
        f = line.split()
        if f and f[0] == "isjl":
            pinned[int(f[1])] = float(f[7])
        elif f and f[0] == "ljf":
            pinned[0] = float(f[7])
    for al in RS.ALPHAS:
        thr, thr_l, _, viol = PROF[("spec", al)]
        assert thr == pytest.approx(pinned[al], rel=1e-4) and thr_l == pytest.approx(pinned[0], rel=1e-4)
        assert viol == 0
    assert CR.DELTAS[:4] == (0,) + RS.TINY_DELTAS


@pytest.fixture(scope="module")
def opts():
    return {B: RS.opt_table(B) for B in (2, 3)}


@pytest.mark.parametrize("name", ["spec", "waiver", "short_packs"])
def test_tiny_rows_rederived(name, opts):
    flags = dict(RS.STUDY)[name]
    for B, d, m34, mg, worst, viol in RS.tiny_rows(flags, opts):
        g = TINY[(name, B, d)]
        assert (m34, mg, viol) == (g[0], g[1], g[3]) and worst == pytest.approx(g[2], abs=1e-4)


def test_profit_rows_rederived_on_a_prefix():
    """A 20-replication re-run of two variants: the specified reading keeps
    Eq. 1 on every step, the ungated one breaks it on every replication."""
    for name in ("spec", "ungated_plan"):
        rows = RS.profit_rows(dict(RS.STUDY)[name], reps=20)
        for al, thr, thr_l, ext, viol in rows:
            assert thr > 0 and thr_l > 0 and 0 <= ext <= (10.0 if name == "ungated_plan" else 1.0)
            assert (viol == 0) == (name == "spec")


def test_no_fair_reading_reaches_table1():
    table1 = _table1_isjl_throughput()
    fair = {name for (name, _), v in PROF.items() if v[3] == 0}
    fair = {n for n in fair if all(PROF[(n, al)][3] == 0 for al in RS.ALPHAS)}
    assert {"spec", "waiver", "short_packs", "cancel", "p2_reserved", "literal_long"} <= fair
    for name in fair:
        for al in RS.ALPHAS:
            thr, thr_l, ext, _ = PROF[(name, al)]
            assert ext <= 1.0                       # mean extent within the budget
            assert thr < table1[al] - 1.0, (name, al)   # Table 1 is out of reach
            assert thr < thr_l + 0.1, (name, al)        # and none beats LJF beyond noise
    # dropping the gate on plan entries breaks Eq. 1 on (almost) every replication
    for al in RS.ALPHAS:
        thr, _, _, viol = PROF[("ungated_plan", al)]
        assert viol >= 0.9 * RS.REPS and thr < table1[al]
