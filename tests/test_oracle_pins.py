"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a closed
form the paper proves, a textbook algorithm the method reduces to, an exact
identity of the cost model, a hand-derived schedule, or brute force.
"""
import heapq
import itertools
import math
import os

import numpy as np
import pytest

INF = 2**31 - 1
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def parse_examples(path):
    ex, cur = [], None
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        key, *vals = line.split()
        if key == "name":
            cur = {"name": vals[0]}
        elif key == "policy":
            cur["policy"] = vals[0]
            kv = dict(zip(vals[1::2], vals[2::2]))
            cur["B"] = int(kv["B"])
            cur["delta"] = INF if kv["delta"] == "inf" else int(kv["delta"])
            cur["kv"] = INF if kv["kv"] == "inf" else int(kv["kv"])
        elif key == "end":
            ex.append(cur)
        else:
            cur[key] = np.array([int(v) for v in vals], np.int32)
    return ex


EXAMPLES = parse_examples(os.path.join(GOLDEN, "worked_examples.txt"))


@pytest.mark.parametrize("ex", EXAMPLES, ids=[e["name"] for e in EXAMPLES])
def test_hand_derived_schedules(oracle_mod, ex):
    z = np.zeros_like(ex["o"])
    rec, st, co = oracle_mod.run(ex["policy"], ex["B"], ex["delta"], ex["kv"], ex["arrival"], z, ex["o"],
                                 slack=ex.get("slack"))
    assert rec["status"] == 0
    np.testing.assert_array_equal(st, ex["start"])
    np.testing.assert_array_equal(co, ex["completion"])


# -- Proposition "FCFS can have quadratic batching externality" ------------
@pytest.mark.parametrize("L", list(range(1, 41)) + [97, 250, 1000])
def test_fcfs_quadratic_externality(oracle_mod, L):
    """B=2, one length-L request first, then L unit requests (Sec. 5)."""
    o = np.ones(L + 1, np.int32)
    o[0] = L
    z = np.zeros(L + 1, np.int32)
    r, _, _ = oracle_mod.run("fcfs", 2, INF, INF, z, z, o)
    assert r["T_make"] == L and r["E"] == L * (L - 1) // 2
    r2, _, _ = oracle_mod.run("ljf", 2, INF, INF, z, z, o)
    assert r2["T_make"] == L + math.ceil((L - 1) / 2) and r2["E"] == 0
    # profit gap of Eq. ljf-fcfs-profit-adversarial, in the same fp64 terms
    c, tau = 0.0005, 1e-6
    lhs = r2["profit"] - r["profit"]
    rhs = tau * L * (L - 1) / 2 - c * math.ceil((L - 1) / 2)
    assert abs(lhs - rhs) <= 1e-9 * max(1.0, abs(rhs))


# -- LJF: Algorithm 1 makespan T = o_1 + o_{B+1} + o_{2B+1} + ... ----------
@pytest.mark.parametrize("B", [1, 2, 3, 5, 8])
def test_ljf_closed_form_and_zero_externality(oracle_mod, B):
    rng = np.random.default_rng(11 + B)
    for _ in range(40):
        n = int(rng.integers(1, 40))
        o = rng.integers(1, 60, n).astype(np.int32)
        z = np.zeros(n, np.int32)
        r, _, _ = oracle_mod.run("ljf", B, 0, INF, z, z, o)
        srt = np.sort(o)[::-1]
        assert r["T_make"] == int(srt[::B].sum())           # Thm. LJF proof, T_LJF formula
        assert r["E"] == 0 and r["max_extent"] == 0          # Prop. 1: extent 0
        assert r["violations"] == 0


# -- ISJL at delta = 0 is LJF -----------------------------------------------
def test_isjl_delta0_equals_ljf_offline_any_kv(oracle_mod):
    """theta = 2*0 -> no packs; every long job starts at t0; the gate then
    holds admissions until nothing runs: LJF's static batches."""
    rng = np.random.default_rng(5)
    for _ in range(60):
        n = int(rng.integers(1, 50))
        B = int(rng.integers(1, 9))
        o = rng.integers(1, 40, n).astype(np.int32)
        kv = INF if rng.random() < 0.4 else int(o.max() + rng.integers(0, 80))
        z = np.zeros(n, np.int32)
        r1, s1, c1 = oracle_mod.run("isjl", B, 0, kv, z, z, o)
        r2, s2, c2 = oracle_mod.run("ljf", B, 0, kv, z, z, o)
        np.testing.assert_array_equal(s1, s2)
        np.testing.assert_array_equal(c1, c2)


def test_isjl_delta0_equals_ljf_online_no_kv(oracle_mod):
    rng = np.random.default_rng(6)
    for _ in range(60):
        n = int(rng.integers(1, 50))
        B = int(rng.integers(1, 9))
        o = rng.integers(1, 40, n).astype(np.int32)
        a = np.sort(rng.integers(0, 60, n)).astype(np.int32)
        z = np.zeros(n, np.int32)
        _, s1, _ = oracle_mod.run("isjl", B, 0, INF, a, z, o)
        _, s2, _ = oracle_mod.run("ljf", B, 0, INF, a, z, o)
        np.testing.assert_array_equal(s1, s2)


# -- ISJL at delta = inf is Graham's LPT list scheduling --------------------
def lpt_starts(o, B):
    """Textbook LPT (Graham 1969): longest job first to the earliest free machine."""
    order = sorted(range(len(o)), key=lambda i: (-int(o[i]), i))
    heap = [(0, w) for w in range(B)]
    start = np.zeros(len(o), np.int64)
    for i in order:
        t, w = heapq.heappop(heap)
        start[i] = t
        heapq.heappush(heap, (t + int(o[i]), w))
    return start


@pytest.mark.parametrize("B", [1, 2, 3, 4, 7, 16])
def test_isjl_delta_inf_is_lpt(oracle_mod, B):
    rng = np.random.default_rng(100 + B)
    for _ in range(30):
        n = int(rng.integers(1, 80))
        o = rng.integers(1, 200, n).astype(np.int32)
        z = np.zeros(n, np.int32)
        r, st, co = oracle_mod.run("isjl", B, INF, INF, z, z, o)
        np.testing.assert_array_equal(st, lpt_starts(o, B))
        assert r["T_make"] == int((lpt_starts(o, B) + o).max())


# -- Jigsaw family (Sec. 4.1): T_LPT = 4B-1, T_OPT = 3B ----------------------
def jigsaw(B):
    o = []
    for v in range(2 * B - 1, B, -1):
        o += [v, v]
    o += [B, B, B]
    return np.array(o, np.int32)


@pytest.mark.parametrize("B", [2, 3, 4, 6, 10])
def test_jigsaw_isjl_makespan(oracle_mod, B):
    o = jigsaw(B)
    z = np.zeros_like(o)
    r, _, _ = oracle_mod.run("isjl", B, INF, INF, z, z, o)
    assert r["T_make"] == 4 * B - 1


@pytest.mark.parametrize("B", [2, 3])
def test_jigsaw_opt(oracle_mod, B):
    o = jigsaw(B)
    assert oracle_mod.opt_makespan(np.zeros_like(o), o, B, INF) == 3 * B


# -- Online two-request adversary (Prop. online lower bound) ----------------
@pytest.mark.parametrize("L,alpha", [(12, 0), (20, 3), (30, 5), (40, 10)])
def test_online_two_request_adversary(oracle_mod, L, alpha):
    """J1 of length L at time 0; J2 of length L released at alpha+1 (s = 0)."""
    a = np.array([0, alpha + 1], np.int32)
    o = np.array([L, L], np.int32)
    z = np.zeros(2, np.int32)
    r, st, _ = oracle_mod.run("isjl", 2, alpha, INF, a, z, o)
    assert st[0] == 0 and r["T_make"] == 2 * L             # T_A >= s + 2L
    assert oracle_mod.opt_makespan(a, o, 2, alpha) == L + alpha + 1   # wait, start together


# -- Exact identities of the cost model (Theorem "Profit decomposition") ----
def _small_instances(rng, count, online):
    for _ in range(count):
        n = int(rng.integers(1, 120))
        p = rng.integers(0, 40, n).astype(np.int32)
        out = rng.integers(1, 120, n).astype(np.int32)
        a = (np.sort(rng.integers(0, 300, n)) if online else np.zeros(n)).astype(np.int32)
        yield a, p, out


@pytest.mark.parametrize("online", [False, True])
def test_cost_identities_and_invariants(oracle_mod, online):
    rng = np.random.default_rng(21 + online)
    for a, p, out in _small_instances(rng, 40, online):
        o = p.astype(np.int64) + out
        B = int(rng.integers(1, 12))
        kv = INF if rng.random() < 0.3 else int(o.max() + rng.integers(0, 400))
        Q = int((o * (o + 1) // 2).sum())
        recs = {}
        for pol, d in [("fcfs", 0), ("ljf", 0)] + [("isjl", d) for d in (0, 1, 7, 30, INF)]:
            r, st, co = oracle_mod.run(pol, B, d, kv, a, p, out)
            assert r["status"] == 0
            assert r["Q"] == Q and r["O"] == int(o.sum())
            assert r["W"] == r["Q"] + r["E"]                 # sum_t sum_S r_i = Q
            assert r["token_adv"] == r["O"]                  # sum_t |S(t)| = O
            assert r["kv_violations"] == 0 and r["peak_kv"] <= kv
            assert r["peak_batch"] <= B
            np.testing.assert_array_equal(co - st, o)        # contiguous service
            assert (st >= a).all()
            assert r["sum_completion"] == int(co.sum())
            assert r["sum_latency"] == int((co - a).sum())
            assert r["T_make"] == int(co.max())
            if pol != "fcfs":
                assert r["violations"] == 0                  # Eq. 1 at every step
                if d != INF:
                    assert r["E"] <= d * r["O"]              # E <= alpha * O
            assert r["revenue"] == 0.002 * float(o.sum())    # policy-independent
            recs[(pol, d)] = r
        # pairwise identity Pi_A - Pi_B = c(T_B - T_A) + tau(E_B - E_A)
        keys = list(recs)
        for k1, k2 in zip(keys, keys[1:]):
            A, Bb = recs[k1], recs[k2]
            lhs = A["profit"] - Bb["profit"]
            rhs = 0.0005 * (Bb["T_busy"] - A["T_busy"]) + 1e-6 * (Bb["E"] - A["E"])
            assert abs(lhs - rhs) <= 1e-9 * max(1.0, abs(A["cost"]))


def test_fcfs_is_arrival_order(oracle_mod):
    """FCFS never lets a later request start before an earlier one."""
    rng = np.random.default_rng(3)
    for a, p, out in _small_instances(rng, 30, True):
        B = int(rng.integers(1, 6))
        kv = int((p + out).max() + rng.integers(0, 200))
        _, st, _ = oracle_mod.run("fcfs", B, 0, kv, a, p, out)
        assert (np.diff(st) >= 0).all()


# -- The offline optimum ------------------------------------------------------
def pcmax_bruteforce(o, B):
    best = None
    for assign in itertools.product(range(B), repeat=len(o)):
        loads = [0] * B
        for i, m in enumerate(assign):
            loads[m] += int(o[i])
        v = max(loads)
        best = v if best is None else min(best, v)
    return best


@pytest.mark.parametrize("B", [1, 2, 3])
def test_opt_without_fairness_is_pcmax(oracle_mod, B):
    rng = np.random.default_rng(40 + B)
    for _ in range(25):
        n = int(rng.integers(1, 7))
        o = rng.integers(1, 13, n).astype(np.int32)
        assert oracle_mod.opt_makespan(np.zeros(n, np.int32), o, B, INF) == pcmax_bruteforce(o, B)


@pytest.mark.parametrize("B", [1, 2, 3])
def test_opt_at_delta0_is_ljf(oracle_mod, B):
    """alpha = 0: co-running jobs have equal progress, so the schedule is a
    sequence of batches; sorted consecutive grouping minimises the sum of
    batch maxima."""
    rng = np.random.default_rng(50 + B)
    for _ in range(25):
        n = int(rng.integers(1, 7))
        o = rng.integers(1, 13, n).astype(np.int32)
        srt = np.sort(o)[::-1]
        assert oracle_mod.opt_makespan(np.zeros(n, np.int32), o, B, 0) == int(srt[::B].sum())


def test_opt_nested_frontier(oracle_mod):
    """Prop. nested alpha frontier: T*_alpha is non-increasing in alpha."""
    rng = np.random.default_rng(60)
    for _ in range(30):
        n = int(rng.integers(2, 7))
        B = int(rng.integers(2, 4))
        o = rng.integers(1, 13, n).astype(np.int32)
        z = np.zeros(n, np.int32)
        ts = [oracle_mod.opt_makespan(z, o, B, d) for d in (0, 1, 2, 4, 8, INF)]
        assert all(x >= y for x, y in zip(ts, ts[1:]))
        # and OPT never loses to any simulated fair policy
        for d in (0, 2, INF):
            r, _, _ = oracle_mod.run("isjl", B, d, INF, z, z, o)
            assert oracle_mod.opt_makespan(z, o, B, d) <= r["T_make"]


# -- Validation and the step guard -------------------------------------------
def test_oracle_errors(oracle_mod):
    z = np.zeros(3, np.int32)
    o = np.array([3, 2, 1], np.int32)
    assert oracle_mod.run("fcfs", 2, 0, 2, z, z, o)[0]["status"] == 2        # o > kv_cap
    assert oracle_mod.run("fcfs", 2, 0, INF, z, z, np.array([3, 0, 1], np.int32))[0]["status"] == 2
    assert oracle_mod.run("fcfs", 2, 0, INF, np.array([0, 2, 1], np.int32), z, o)[0]["status"] == 1
    assert oracle_mod.run("fcfs", 2, 0, INF, z, np.array([0, -1, 0], np.int32), o)[0]["status"] == 1
    assert oracle_mod.run("fcfs", 0, 0, INF, z, z, o)[0]["status"] == 1
    assert oracle_mod.run("isjl", 2, 0, INF, z, z, o, max_steps=2)[0]["status"] == 5


@pytest.mark.parametrize("policy", ["isjl", "isjl_beta"])
def test_b2_first_stage_follows_the_stage_definition(oracle_mod, policy):
    """B = 2, all requests at t = 0, o_2 > alpha: the first stage is the one
    the proof of Theorem "Competitive ratio of Algorithm ISJL" defines (its
    "stage" definition): the pack P runs alone for P - alpha steps (if
    positive), L = o_1 joins it until P ends, then S = o_2 starts beside L.
    The pack is the B = 2 rule of Section 3.2: scanning the shorter requests
    longest first, take each that keeps the pack within
    q = min{o_1 - o_2 + beta, 2 alpha} (beta = alpha for Algorithm 2)."""
    O = oracle_mod
    rng = np.random.default_rng(31 if policy == "isjl" else 32)
    checked = 0
    for _ in range(400):
        n = int(rng.integers(3, 12))
        o = rng.integers(1, 60, n).astype(np.int32)
        alpha = int(rng.integers(1, 30))
        order = sorted(range(n), key=lambda i: (-int(o[i]), i))
        o1, o2 = int(o[order[0]]), int(o[order[1]])
        if o2 <= alpha:
            continue
        beta = alpha if policy == "isjl" else O.beta(alpha)
        q = min(o1 - o2 + beta, 2 * alpha)
        pack, P = [], 0
        for i in order[2:]:
            if P + int(o[i]) <= q:
                pack.append(i)
                P += int(o[i])
        _, st, co = O.run(policy, 2, alpha, INF, np.zeros(n, np.int32), np.zeros(n, np.int32), o)
        t = 0
        for i in pack:                     # the pack runs back to back from step 0
            assert st[i] == t, (o, alpha, pack)
            t += int(o[i])
        assert st[order[0]] == max(P - alpha, 0)     # L joins after P - alpha steps
        assert st[order[1]] == P                     # S starts when the pack ends
        # Phase TWO at the first freed worker (Section 3.2): the longest
        # unprocessed request starts there if the other worker's decode length
        # is at most alpha, else not before the other one ends
        endL, endS = int(co[order[0]]), int(co[order[1]])
        rest = [i for i in order[2:] if i not in pack]
        if rest and endL != endS:
            t1, other_start, other_end = ((endL, P, endS) if endL < endS else (endS, st[order[0]], endL))
            nxt = rest[0]
            if t1 - other_start <= alpha:
                assert st[nxt] == t1, (o, alpha)
            else:
                assert st[nxt] >= other_end, (o, alpha)
        checked += 1
    assert checked > 100


@pytest.mark.parametrize("B", [3, 4, 6])
def test_first_stage_timing_with_short_packs(oracle_mod, B):
    """B >= 3, all requests at t = 0, at most B requests longer than alpha and
    the rest at most alpha long: Algorithm 2's first stage as Section 3.3
    describes it.  Each pack runs back to back from step 0 on its worker (a
    pack member of length <= alpha can never shut the gate), o_1 is held back
    d1 = min{max{max_j sum(w_j) - alpha, 0}, alpha} steps, and each long
    request o_j (2 <= j <= M) starts on its worker when its pack has ended,
    and not before o_1.  Packs: each shorter request, longest first, goes to
    the first worker with room, visiting the workers without a long request
    (budget alpha) in order, then the workers of o_M, ..., o_2 (budget
    min{2 alpha, o_1 - o_j + alpha})."""
    O = oracle_mod
    rng = np.random.default_rng(40 + B)
    checked = 0
    for _ in range(300):
        alpha = int(rng.integers(2, 25))
        n_long = int(rng.integers(2, B + 1))
        n_short = int(rng.integers(0, 3 * B))
        o = np.concatenate([rng.integers(alpha + 1, 4 * alpha + 2, n_long),
                            rng.integers(1, alpha + 1, n_short)]).astype(np.int32)
        o = o[rng.permutation(len(o))]
        n = len(o)
        order = sorted(range(n), key=lambda i: (-int(o[i]), i))
        M = n_long
        o1 = int(o[order[0]])
        budget = {j: alpha for j in range(M + 1, B + 1)}
        budget.update({j: min(2 * alpha, o1 - int(o[order[j - 1]]) + alpha) for j in range(2, M + 1)})
        visit = list(range(M + 1, B + 1)) + list(range(M, 1, -1))
        packs = {j: [] for j in visit}
        for i in order[M:]:
            for j in visit:
                if sum(int(o[x]) for x in packs[j]) + int(o[i]) <= budget[j]:
                    packs[j].append(i)
                    break
        sums = {j: sum(int(o[x]) for x in packs[j]) for j in visit}
        d1 = min(max(max(sums[j] for j in range(2, M + 1)) - alpha, 0), alpha)
        _, st, _ = O.run("isjl", B, alpha, INF, np.zeros(n, np.int32), np.zeros(n, np.int32), o)
        for j in visit:
            t = 0
            for i in packs[j]:
                assert st[i] == t, (o.tolist(), alpha, j)
                t += int(o[i])
        assert st[order[0]] == d1, (o.tolist(), alpha)
        for j in range(2, M + 1):
            assert st[order[j - 1]] == max(sums[j], d1), (o.tolist(), alpha, j)
        checked += 1
    assert checked == 300
