"""ISJL against the exhaustive offline optimum on the tiny-exhaustive workload.

Theorem "Competitive ratio of Algorithm ISJL" (B = 2) and Theorem "Competitive
ratio of Algorithm 2" (B >= 2) claim T_OPT / T_ISJL >= 3/4 offline with no KV
cap.  For B = 2 the oracle meets it, and the sharper CR(gamma) bound, on all
4096 instances.  For B = 3 it misses both on the instances listed in
tests/golden/cr_findings.txt (a finding about Algorithm 2's generalisation,
recorded, not hidden); this test pins that exact list.
"""
import os
import sys

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))
import make_cr_findings as F  # noqa: E402

INF = 2**31 - 1


def load_findings():
    out = {}
    for line in open(os.path.join(HERE, "golden", "cr_findings.txt")):
        if line.startswith("#") or not line.strip():
            continue
        B, d, bound, cnt, *ids = line.split()
        d = INF if d == "inf" else int(d)
        out[(int(B), d, bound)] = [int(x) for x in ids]
        assert len(ids) == int(cnt)
    return out


@pytest.fixture(scope="module")
def computed():
    return F.compute()


def test_b2_meets_three_quarters_and_gamma(computed):
    for d in F.DELTAS:
        f34, fg = computed[(2, d)]
        assert f34 == [] and fg == [], (d, f34[:5], fg[:5])


def test_b3_misses_match_recorded_findings(computed):
    rec = load_findings()
    for d in F.DELTAS:
        f34, fg = computed[(3, d)]
        assert f34 == rec[(3, d, "3/4")]
        assert fg == rec[(3, d, "gamma")]
    # the bound holds at both ends of the budget range
    assert computed[(3, 0)] == ([], []) and computed[(3, INF)] == ([], [])


def test_b2_isjl_with_optimal_beta_meets_its_bound():
    """Theorem "Competitive ratio of Algorithm ISJL" (B = 2): with
    beta = (sqrt(17) - 1)/4 alpha, T_OPT / T >= min{(a + 2b)/(a + 3b), 4a/(6a - b)}
    (about 0.766), on every tiny instance, offline without a KV cap."""
    import math
    from oracle import oracle as O
    from paper_2608_02244_gb300 import workloads as W
    a, p, out = W.generate(2)
    o = p + out
    for d in (1, 2, 4, 8):
        beta = (math.sqrt(17) - 1) / 4 * d
        bound = min((d + 2 * beta) / (d + 3 * beta), 4 * d / (6 * d - beta))
        rec, _, _ = O.run("isjl_beta", 2, d, INF, a, p, out, per_request=False)
        assert (rec["violations"] == 0).all()
        for i in range(len(o)):
            assert O.opt_makespan(a[i], o[i], 2, d) >= bound * rec["T_make"][i] - 1e-9, (d, i)


def test_ljf_and_lpt_bounds_against_the_unconstrained_optimum():
    """Theorem "Competitive Ratio of Algorithm LJF": T_OPT / T_LJF >= B / (2B - 1),
    and Graham's bound for list scheduling longest first (the proposition the
    proofs use for Phase TWO; ISJL at alpha = infinity is that rule):
    T_OPT / T_ISJL(inf) >= 3B / (4B - 1); T_OPT without the fairness
    constraint, every tiny instance, B = 2 and 3.  The LJF bound is attained by
    o = (2, 1, 1) with B = 2: LJF needs 3 steps, the optimum 2."""
    import numpy as np
    from oracle import oracle as O
    from paper_2608_02244_gb300 import workloads as W
    a, p, out = W.generate(2)
    o = p + out
    for B in (2, 3):
        ljf, _, _ = O.run("ljf", B, 0, INF, a, p, out, per_request=False)
        lpt, _, _ = O.run("isjl", B, INF, INF, a, p, out, per_request=False)
        for i in range(len(o)):
            T = O.opt_makespan(a[i], o[i], B, INF)
            assert T * (2 * B - 1) >= B * int(ljf["T_make"][i]), (B, i)
            assert T * (4 * B - 1) >= 3 * B * int(lpt["T_make"][i]), (B, i)
    z = np.zeros((1, 3), np.int32)
    out3 = np.array([[2, 1, 1]], np.int32)
    rec, _, _ = O.run("ljf", 2, 0, INF, z, z, out3, per_request=False)
    assert int(rec["T_make"][0]) == 3 and O.opt_makespan(z[0], out3[0], 2, INF) == 2
