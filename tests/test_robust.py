"""Robust-ISJL (Section 3.3): planning with upper-bound predictions u_i = o_i + e_i.

Pins: with zero slack every policy equals its clairvoyant run; the fairness
constraint (Theorem "Fairness of Robust-ISJL") and the KV reservation hold on
every step; Theorem "Competitive guarantee of Robust-ISJL under interval
uncertainty", T <= 4/3 (T_OPT + Delta^pack), and its scale-normalised
corollary hold on the tiny-robust instances except the recorded B = 3 miss.
"""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.join(HERE, "golden"))
import make_robust_findings as F  # noqa: E402

INF = 2**31 - 1
POLS = [("fcfs", 0), ("ljf", 0), ("isjl", 3), ("isjl", 25), ("isjl", INF), ("sjf", 0), ("isjl_beta", 25)]


def _instances(rng, count):
    for _ in range(count):
        n = int(rng.integers(1, 90))
        a = np.sort(rng.integers(0, 200, n)).astype(np.int32)
        p = rng.integers(0, 30, n).astype(np.int32)
        o = rng.integers(1, 80, n).astype(np.int32)
        e = rng.integers(0, 40, n).astype(np.int32)
        yield a, p, o, e


def test_zero_slack_is_the_clairvoyant_policy(oracle_mod):
    rng = np.random.default_rng(31)
    for a, p, o, _ in _instances(rng, 25):
        B = int(rng.integers(1, 9))
        kv = int((p + o).max() + rng.integers(0, 300))
        z = np.zeros_like(a)
        for pol, d in POLS:
            r1, s1, c1 = oracle_mod.run(pol, B, d, kv, a, p, o)
            r2, s2, c2 = oracle_mod.run(pol, B, d, kv, a, p, o, slack=z)
            assert r1.tobytes() == r2.tobytes()
            np.testing.assert_array_equal(s1, s2)
            np.testing.assert_array_equal(c1, c2)


def test_fairness_and_kv_reservation_with_predictions(oracle_mod):
    rng = np.random.default_rng(32)
    for a, p, o, e in _instances(rng, 25):
        B = int(rng.integers(1, 9))
        u = p.astype(np.int64) + o + e
        kv = int(u.max() + rng.integers(0, 300))
        for pol, d in POLS:
            r, st, co = oracle_mod.run(pol, B, d, kv, a, p, o, slack=e)
            assert r["status"] == 0
            np.testing.assert_array_equal(co - st, p + o)          # true lengths are served
            assert r["peak_kv"] <= kv and r["kv_violations"] == 0   # reservations of u_i fit
            assert r["W"] == r["Q"] + r["E"] and r["token_adv"] == r["O"]
            if pol not in ("fcfs", "sjf"):
                assert r["violations"] == 0                         # gate on true progress


def test_infeasible_when_prediction_exceeds_kv_cap(oracle_mod):
    z = np.zeros(2, np.int32)
    r, _, _ = oracle_mod.run("isjl", 2, 4, 10, z, z, np.array([5, 5], np.int32), slack=np.array([0, 6], np.int32))
    assert r["status"] == 2
    r, _, _ = oracle_mod.run("isjl", 2, 4, 10, z, z, np.array([5, 5], np.int32), slack=np.array([0, -1], np.int32))
    assert r["status"] == 1


def _recorded():
    out = {}
    for line in open(os.path.join(HERE, "golden", "robust_findings.txt")):
        if line.startswith("#") or not line.strip():
            continue
        left, right = line.split("|")
        B, d, cnt, *ids = left.split()
        out[(int(B), INF if d == "inf" else int(d))] = ([int(x) for x in ids], int(right))
    return out


def test_robust_guarantee_b2():
    rec = _recorded()
    for d in (0, 1, 2, 4, INF):
        thm, cor, viol = F.misses(2, d, list(range(1024)))
        assert thm == [] and cor == [] and viol == 0, d
        assert rec[(2, d)] == ([], 0)


def test_robust_guarantee_b3_recorded_miss():
    """B = 3, alpha = 4: the one miss (Algorithm 2's B = 3 misses carry over)."""
    rec = _recorded()
    thm, cor, viol = F.misses(3, 4)
    assert (thm, len(cor)) == rec[(3, 4)] and viol == 0
