"""The oracle's records against a recount from its own schedules.

For every request the oracle reports when it started and completed.  From
those steps alone the model fixes everything else (Section 2: a request runs
contiguously, one token per step, r_i = steps it has run including the
current one; Section 5: a nonempty step costs |S| max r, E adds max r - r_i
per running request; extent = max r - min r).  This recount is a second,
independent statement of the accounting, so a slip in the oracle's per-step
bookkeeping (W, E, extent, T_busy, T_make, completion sums, KV peak) fails
here on random instances of every policy, with and without arrivals, a KV
cap, upper-bound slack and a fairness budget.  It also checks what the
policies promise: contiguous service of exactly o_i tokens, no start before
the arrival, at most B running, the reserved KV within the cap, and Eq. 1 on
every step for LJF and ISJL.
"""
import numpy as np
import pytest

INF = 2**31 - 1


def recount(a, o, u, st, co, kv_cap):
    """Per-step recount from the schedule: o true lengths, u planning lengths
    (KV reservation), st / co start and completion steps."""
    T_make = int(co.max())
    W = E = busy = sum_ext = max_ext = tok = 0
    peak_kv = peak_b = 0
    exts = []
    for k in range(T_make):
        run = np.nonzero((st <= k) & (k < co))[0]
        if run.size == 0:
            continue
        r = k - st[run] + 1                      # token processed in step k
        m = int(r.max())
        W += run.size * m
        E += int((m - r).sum())
        ext = m - int(r.min())
        exts.append(ext)
        sum_ext += ext
        max_ext = max(max_ext, ext)
        busy += 1
        tok += run.size
        peak_kv = max(peak_kv, int(u[run].sum()))
        peak_b = max(peak_b, run.size)
    return dict(T_make=T_make, T_busy=busy, W=W, E=E, sum_extent=sum_ext, max_extent=max_ext,
                token_adv=tok, peak_kv=peak_kv, peak_batch=peak_b, sum_completion=int(co.sum()),
                sum_latency=int((co - a).sum()), exts=exts)


@pytest.mark.parametrize("policy", ["fcfs", "ljf", "sjf", "isjl", "isjl_beta"])
def test_records_equal_recount_from_schedule(oracle_mod, policy):
    O = oracle_mod
    rng = np.random.default_rng(["fcfs", "ljf", "sjf", "isjl", "isjl_beta"].index(policy) + 77)
    for case in range(120):
        n = int(rng.integers(1, 14))
        B = int(rng.integers(1, 6))
        if case % 3 == 0:
            a = np.zeros(n, np.int32)
        else:
            a = np.sort(rng.integers(0, 25, n)).astype(np.int32)
        o = rng.integers(1, 22, n).astype(np.int32)
        e = rng.integers(0, 6, n).astype(np.int32) if case % 4 == 0 else None
        u = o + (e if e is not None else 0)
        kv = INF if case % 2 == 0 else int(rng.integers(int(u.max()), int(u.max()) * 3 + 1))
        alpha = [0, 1, 2, 3, 5, 8, 13, INF][case % 8]
        rec, st, co = O.run(policy, B, alpha, kv, a, np.zeros(n, np.int32), o, slack=e)
        assert rec["status"] == 0
        # the schedule itself: contiguous service of o_i tokens after the arrival
        assert (st >= a).all() and (co - st == o).all()
        got = recount(a, o, u, st, co, kv)
        for f in ("T_make", "T_busy", "W", "E", "sum_extent", "max_extent", "token_adv", "peak_kv",
                  "peak_batch", "sum_completion", "sum_latency"):
            assert int(rec[f]) == got[f], (policy, case, f, int(rec[f]), got[f])
        assert got["peak_batch"] <= B and got["peak_kv"] <= kv
        assert int(rec["violations"]) == sum(x > alpha for x in got["exts"])
        if policy in ("ljf", "isjl", "isjl_beta"):
            assert int(rec["violations"]) == 0 and got["max_extent"] <= alpha
