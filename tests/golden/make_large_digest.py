"""Write tests/golden/large_instance_digest.txt: per-instance digests of the
oracle's results on the whole large-instance workload.

The workload (1,024 instances x 100,000 requests, Poisson arrivals with mean
gap 0.05, B = 512, KV cap 1,000,000) runs under FCFS, LJF and ISJL with
delta = 256.  The oracle needs about ten seconds per instance for the three
runs, too long for a test run, so this script runs it once on every host core
and stores, per instance:

  input digest   over the generated arrival, prompt and output arrays, so a
                 test can tell whether its platform drew the same inputs;
  result digest  over the integer record fields (oracle.RECORD_FIELDS_I64, as
                 int64) and the per-request start and completion steps (int32)
                 of the three runs, in run order.

Both digests are BLAKE2b with an 8-byte output over little-endian bytes.  Only
the oracle, the workload generator and numpy are used.

    python tests/golden/make_large_digest.py [processes]
"""
from __future__ import annotations

import hashlib
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from oracle import parallel  # noqa: E402
from paper_2608_02244_gb300 import workloads as W  # noqa: E402

WID = 5
RUNS = [("fcfs", 0), ("ljf", 0), ("isjl", 256)]
OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "large_instance_digest.txt")
BLOCK = 64          # instances generated and simulated at a time (bounds host memory)


def input_digest(a, p, o) -> str:
    h = hashlib.blake2b(digest_size=8)
    for x in (a, p, o):
        h.update(np.ascontiguousarray(x, dtype="<i4").tobytes())
    return h.hexdigest()


def result_digest(recs, starts, compls) -> str:
    """recs: one record per run; starts / compls: one int32 row per run."""
    h = hashlib.blake2b(digest_size=8)
    for r, st, co in zip(recs, starts, compls):
        h.update(np.array([r[f] for f in O.RECORD_FIELDS_I64], dtype="<i8").tobytes())
        h.update(np.ascontiguousarray(st, dtype="<i4").tobytes())
        h.update(np.ascontiguousarray(co, dtype="<i4").tobytes())
    return h.hexdigest()


def main() -> None:
    procs = int(sys.argv[1]) if len(sys.argv) > 1 else None
    wl = W.WORKLOADS[WID]
    B, kv = wl.B[0], wl.kv_caps[0]
    pool = parallel.make_pool(procs)
    lines = []
    totals = {pol: np.zeros(4, np.int64) for pol, _ in RUNS}
    t0 = time.time()
    for s in range(0, wl.n_instances, BLOCK):
        ids = range(s, min(wl.n_instances, s + BLOCK))
        a, p, o = W.generate(WID, instances=ids)
        res = [parallel.run(pool, pol, B, d, kv, a, p, o, per_request=True, block=1) for pol, d in RUNS]
        for k, i in enumerate(ids):
            recs = [r[0][k] for r in res]
            lines.append(f"{i} {input_digest(a[k], p[k], o[k])} "
                         f"{result_digest(recs, [r[1][k] for r in res], [r[2][k] for r in res])}")
        for (pol, _), r in zip(RUNS, res):
            totals[pol] += np.array([r[0][f].sum() for f in ("T_busy", "W", "E", "sum_completion")], np.int64)
        print(f"{ids[-1] + 1} / {wl.n_instances} instances, {time.time() - t0:.0f} s", flush=True)
    pool.close()
    pool.join()
    with open(OUT, "w") as f:
        f.write("# Oracle digests of the large-instance workload (1,024 x 100,000 requests, Poisson\n"
                "# arrivals with mean gap 0.05, B = 512, KV cap 1,000,000), runs FCFS, LJF and ISJL\n"
                "# delta = 256.  Written by make_large_digest.py (oracle and workload generator only).\n"
                "# totals <policy> <delta>: sums over the instances of T_busy, W, E, sum_completion\n")
        for pol, d in RUNS:
            f.write(f"# totals {pol} {d} " + " ".join(str(int(x)) for x in totals[pol]) + "\n")
        f.write("# columns: instance input_digest result_digest\n")
        f.write("\n".join(lines) + "\n")
    print(f"wrote {OUT} in {time.time() - t0:.0f} s")


if __name__ == "__main__":
    main()
