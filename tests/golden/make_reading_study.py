"""Write tests/golden/isjl_reading_study.txt: Algorithm 2 under alternative
readings of the passages the paper leaves open, measured against what the
paper fixes.

Each variant switches one reading of the oracle's ISJL away from the
specified one (the oracle's VARIANTS flags; 0 is the specification).  For
every variant the file records

  - the profit experiment of Section 5.2 (first 200 replications of the
    profit-experiment workload, B = 50, no KV cap), per alpha: mean
    throughput O / T_make next to LJF's, mean average extent / alpha, and
    how many replications break Eq. 1 (a step with extent > alpha);
  - the tiny-exhaustive workload (4096 instances of n = 6, no KV cap), per
    B in {2, 3} and delta in {1, 2, 4}: instances missing the 3/4 bound of
    Theorem "Competitive ratio of Algorithm 2", instances missing the
    CR(gamma) bound of Theorem "Generalized global competitive ratio", the
    worst T_OPT / T_ISJL, and instances with an Eq. 1 violation.

Only the oracle and numpy compute anything here.

Usage: python tests/golden/make_reading_study.py
"""
from __future__ import annotations

import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, HERE)

from oracle import oracle as O  # noqa: E402
from paper_2608_02244_gb300 import workloads as W  # noqa: E402
import make_cr_findings as CR  # noqa: E402

INF = 2**31 - 1
REPS = 200
ALPHAS = W.WORKLOADS[6].deltas
TINY_DELTAS = (1, 2, 4)
V = O.VARIANTS
# one reading switched at a time, plus the contrast that drops the gate on plan entries
STUDY = [
    ("spec", 0),
    ("waiver", V["waiver"]),
    ("no_wait_o1", V["no_wait_o1"]),
    ("d1_last", V["d1_last"]),
    ("p2_reserved", V["p2_reserved"]),
    ("rebuild_reopen", V["rebuild_reopen"]),
    ("literal_long", V["literal_long"]),
    ("short_packs", V["short_packs"]),
    ("cancel", V["cancel"]),
    ("ungated_plan", V["ungated_plan"]),
]


def profit_rows(flags, reps=REPS):
    a, p, o, cnt = W.generate(6, reps, with_counts=True)
    ljf, _, _ = O.run("ljf", 50, 0, INF, a, p, o, per_request=False, counts=cnt)
    rows = []
    for al in ALPHAS:
        r, _, _ = O.run("isjl", 50, al, INF, a, p, o, per_request=False, counts=cnt, variant=flags)
        ext = r["sum_extent"] / np.maximum(r["T_busy"], 1)
        rows.append((al, float(np.mean(r["throughput"])), float(np.mean(ljf["throughput"])),
                     float(np.mean(ext)) / al, int((r["violations"] > 0).sum())))
    return rows


def opt_table(B, deltas=TINY_DELTAS):
    a, p, out = W.generate(2)
    o = p + out
    return {d: np.array([O.opt_makespan(a[i], o[i], B, d) for i in range(len(o))]) for d in deltas}


def tiny_rows(flags, opts):
    a, p, out = W.generate(2)
    o = p + out
    rows = []
    for B in (2, 3):
        for d in TINY_DELTAS:
            r, _, _ = O.run("isjl", B, d, INF, a, p, out, per_request=False, variant=flags)
            T = r["T_make"]
            m34 = mg = 0
            worst = 1.0
            for i in range(len(o)):
                x, y = CR.misses(int(opts[B][d][i]), int(T[i]), int(o[i].max()), d)
                m34 += x
                mg += y
                worst = min(worst, opts[B][d][i] / T[i])
            rows.append((B, d, m34, mg, worst, int((r["violations"] > 0).sum())))
    return rows


def main():
    opts = {B: opt_table(B) for B in (2, 3)}
    path = os.path.join(HERE, "isjl_reading_study.txt")
    with open(path, "w") as f:
        f.write("# Algorithm 2 under alternative readings (oracle only; written by make_reading_study.py).\n"
                "# profit lines: variant 'profit' alpha thr_isjl thr_ljf extent_over_alpha reps_breaking_eq1"
                f"   ({REPS} replications, B = 50)\n"
                "# tiny lines:   variant 'tiny' B delta misses_3/4 misses_gamma worst_ratio instances_breaking_eq1"
                "   (4096 instances, n = 6)\n")
        for name, flags in STUDY:
            for al, thr, thr_l, ext, viol in profit_rows(flags):
                f.write(f"{name} profit {al} {thr:.4f} {thr_l:.4f} {ext:.4f} {viol}\n")
            for B, d, m34, mg, worst, viol in tiny_rows(flags, opts):
                f.write(f"{name} tiny {B} {d} {m34} {mg} {worst:.4f} {viol}\n")
    print(path)


if __name__ == "__main__":
    main()
