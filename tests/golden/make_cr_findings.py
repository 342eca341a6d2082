"""Write tests/golden/cr_findings.txt: where ISJL misses the paper's bounds.

Theorem "Competitive ratio of Algorithm 2" claims T_OPT / T_ISJL >= 3/4 for
every B >= 2 (offline, no KV cap), and Theorem "Generalized global competitive
ratio as a function of gamma" claims the sharper piecewise bound
CR(gamma), gamma = alpha / o_1.  This script runs the CPU oracle's ISJL and
its exhaustive offline optimum on every instance of the tiny-exhaustive
workload (4096 instances of n = 6, o = U[1,4] + U[1,8]) and lists the
instances that miss either bound.  Only the oracle computes anything here.

Usage: python tests/golden/make_cr_findings.py
"""
from __future__ import annotations

import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from paper_2608_02244_gb300 import workloads as W  # noqa: E402

INF = 2**31 - 1
DELTAS = (0, 1, 2, 4, INF)


def misses(T_opt, T_alg, o1, delta):
    """(misses 3/4, misses CR(gamma)) in exact integer arithmetic."""
    m34 = 4 * T_opt < 3 * T_alg
    mg = False
    if 0 < delta < o1:
        if 2 * delta <= o1:      # (1+g)/(1+2g) = (o1+d)/(o1+2d)
            mg = T_opt * (o1 + 2 * delta) < T_alg * (o1 + delta)
        else:                    # (2-g)/(3-2g) = (2 o1 - d)/(3 o1 - 2 d)
            mg = T_opt * (3 * o1 - 2 * delta) < T_alg * (2 * o1 - delta)
    return m34, mg


def compute(kv=INF, Bs=(2, 3)):
    a, p, out = W.generate(2)
    o = p + out
    rows = {}
    for B in Bs:
        for d in DELTAS:
            rec, _, _ = O.run("isjl", B, d, kv, a, p, out, per_request=False)
            f34, fg = [], []
            for i in range(len(o)):
                T = O.opt_makespan(a[i], o[i], B, d, kv)
                m34, mg = misses(T, int(rec["T_make"][i]), int(o[i].max()), d)
                if m34:
                    f34.append(i)
                if mg:
                    fg.append(i)
            rows[(B, d)] = (f34, fg)
    return rows


def main():
    rows = compute()
    path = os.path.join(HERE, "cr_findings.txt")
    with open(path, "w") as f:
        f.write("# Instances of the tiny-exhaustive workload (4096 x n=6, seed 2000, no KV cap)\n"
                "# on which the oracle's ISJL misses a competitive-ratio bound of the paper.\n"
                "# Written by tests/golden/make_cr_findings.py (oracle only).\n"
                "# line: B delta bound count ids...   (bound: 3/4 or gamma)\n")
        for (B, d), (f34, fg) in rows.items():
            ds = "inf" if d == INF else str(d)
            f.write(f"{B} {ds} 3/4 {len(f34)} {' '.join(map(str, f34))}\n".rstrip() + "\n")
            f.write(f"{B} {ds} gamma {len(fg)} {' '.join(map(str, fg))}\n".rstrip() + "\n")
    print(path)


if __name__ == "__main__":
    main()
