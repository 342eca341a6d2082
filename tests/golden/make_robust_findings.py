"""Write tests/golden/robust_findings.txt: tiny-robust instances (workload 7,
no KV cap) on which Robust-ISJL misses Theorem "Competitive guarantee of
Robust-ISJL under interval uncertainty": T <= 4/3 (T_OPT + Delta^pack), with
T_OPT the optimum on the true lengths and Delta^pack the least total of the
largest slack per group over partitions into groups of at most B requests
whose true lengths span at most alpha.  Only the oracle computes anything.

Usage: python tests/golden/make_robust_findings.py
"""
from __future__ import annotations

import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from paper_2608_02244_gb300 import workloads as W  # noqa: E402

INF = 2**31 - 1


def set_partitions(items):
    if not items:
        yield []
        return
    first, rest = items[0], items[1:]
    for part in set_partitions(rest):
        for i in range(len(part)):
            yield part[:i] + [[first] + part[i]] + part[i + 1:]
        yield [[first]] + part


PARTS6 = list(set_partitions(list(range(6))))


def delta_pack(o, e, B, alpha):
    best = None
    for part in PARTS6 if len(o) == 6 else set_partitions(list(range(len(o)))):
        total = 0
        for G in part:
            if len(G) > B or max(o[i] for i in G) - min(o[i] for i in G) > alpha:
                total = None
                break
            total += max(e[i] for i in G)
        if total is not None and (best is None or total < best):
            best = total
    return best


def misses(B, d, instances=None):
    """(theorem misses, corollary misses, Eq. 1 violations) over the given instances."""
    a, p, out, e = W.generate(7, instances, with_slack=True)
    o = p + out
    rec, _, _ = O.run("isjl", B, d, INF, a, p, out, per_request=False, slack=e)
    thm, cor = [], []
    ids = range(len(o)) if instances is None else instances
    for k, i in enumerate(ids):
        T = int(rec["T_make"][k])
        topt = O.opt_makespan(a[k], o[k], B, d)
        if 3 * T > 4 * (topt + delta_pack(o[k], e[k], B, d)):
            thm.append(int(i))
        eps = e[k].sum() / o[k].sum()
        if topt / T < 0.75 / (1 + B * eps) - 1e-12:
            cor.append(int(i))
    return thm, cor, int(rec["violations"].sum())


def main():
    path = os.path.join(HERE, "robust_findings.txt")
    with open(path, "w") as f:
        f.write("# Robust-ISJL misses of T <= 4/3 (T_OPT + Delta^pack) on the tiny-robust workload\n"
                "# (4096 x n=6, seed 7000, slack U{0..3}, no KV cap); written by make_robust_findings.py\n"
                "# line: B delta theorem_misses ids... | corollary_misses\n")
        for B in (2, 3):
            for d in (0, 1, 2, 4, INF):
                thm, cor, _ = misses(B, d)
                ds = "inf" if d == INF else str(d)
                f.write(f"{B} {ds} {len(thm)} {' '.join(map(str, thm))} | {len(cor)}\n")
    print(path)


if __name__ == "__main__":
    main()
