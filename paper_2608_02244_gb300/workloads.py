"""Seeded synthetic request instances for the batched scheduling simulator.

This module only draws input arrays. It holds none of the scheduling model's
arithmetic (not even o_i = prompt + output): both the CUDA path and the CPU
oracle receive the same three int32 arrays per instance and derive everything
else themselves.

Layout: every array has shape (n_instances, n_per_instance), dtype int32,
instance-major (row i is instance i).  Arrivals are non-decreasing along a row.

Instances are generated in independent chunks so that any instance can be
regenerated alone: chunk c of a workload with seed s draws from
``PCG64(SeedSequence([s, c]))``, in the order arrivals, prompts, outputs (and,
for the bimodal mix, the mixture flag and both components).  A chunk holds
``chunk_instances(n)`` consecutive instances (about 2**20 requests).

The five workloads follow the configurations the simulator is measured on:
request lengths o_i = prompt + output are processed one token per step (the
paper's token-step model, Section 2), with Poisson arrivals for the online
configurations (the release-date model of Section 3.4).
"""
from __future__ import annotations

from dataclasses import dataclass, field
import math

import numpy as np

DELTA_INF = 2**31 - 1   # fairness budget "infinity" (the constraint is vacuous)
KV_INF = 2**31 - 1      # no KV-memory cap (the paper's pure compute-bound model)


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: instance shape, distributions and run grid."""
    wid: int
    name: str
    n_instances: int
    n_per_instance: int
    seed: int
    B: tuple            # batch-slot counts the workload is run with
    kv_caps: tuple      # KV caps (tokens) the workload is run with
    deltas: tuple       # ISJL fairness budgets
    policies: tuple = ("fcfs", "ljf", "isjl")
    online: bool = False
    ragged: bool = False  # instances use a variable number of their slots (see counts)
    robust: bool = False  # comes with an upper-bound slack array (length predictions u = o + slack)
    note: str = ""
    c: float = 0.0005   # fixed cost per service step (Section 5 experiment)
    tau: float = 1e-6   # cost per unit of max-driven footprint
    p0: float = 1.0 / 500.0  # unit token price

    @property
    def n_requests(self) -> int:
        return self.n_instances * self.n_per_instance


WORKLOADS = {
    1: Workload(1, "single-200", 1, 200, 0, B=(32,), kv_caps=(2048,), deltas=(32,),
                note="200 requests at t=0; prompt U[1,32]; output 0.7*U[1,16] + 0.3*U[64,256]"),
    2: Workload(2, "tiny-exhaustive", 4096, 6, 2000, B=(2, 3), kv_caps=(16, KV_INF),
                deltas=(0, 1, 2, 4, DELTA_INF), policies=("isjl",),
                note="n=6 at t=0; prompt U[1,4]; output U[1,8]; checked against the offline optimum"),
    3: Workload(3, "online-delta-sweep", 10_000, 1_000, 3000, B=(256,), kv_caps=(200_000,),
                deltas=(16, 64, 256, 1024, DELTA_INF), online=True,
                note="Poisson arrivals, mean gap 2; prompt LN(ln512,1) in [16,4096]; "
                     "output LN(ln256,1.2) in [1,2048]"),
    4: Workload(4, "heavy-tail-mix", 100_000, 500, 4000, B=(128,), kv_caps=(65_536,),
                deltas=(32, 128, 512),
                note="t=0; prompt U[16,1024]; output Pareto(1.5, x_min=8) clipped at 8192"),
    5: Workload(5, "large-instance", 1_024, 100_000, 5000, B=(512,), kv_caps=(1_000_000,),
                deltas=(256,), online=True,
                note="Poisson arrivals, mean gap 0.05; prompt LN(ln1024,1) in [16,32768]; "
                     "output LN(ln512,1.3) in [1,16384]"),
    # Section 5.2: 400 offered requests, o ~ U{1..1000}, price p0 o with p0 = 1/500, and a request in
    # length bucket b = ceil(o / 100) accepts with probability max{0, 1 - o / ((2b - 1) 100)}; the
    # accepted requests (in offer order) form the instance, served with B = 50 and no KV cap.
    6: Workload(6, "profit-experiment", 10_000, 400, 6000, B=(50,), kv_caps=(KV_INF,),
                deltas=(50, 100, 150, 250, 300, 400, 500), ragged=True,
                note="400 offered, o ~ U{1..1000}, bucketed acceptance; accepted requests at t=0"),
    # Section 3.3 (prediction intervals): the instances of workloads 2 and 3 with an upper-bound
    # slack e_i = u_i - o_i drawn per request
    7: Workload(7, "tiny-robust", 4096, 6, 7000, B=(2, 3), kv_caps=(16, KV_INF),
                deltas=(0, 1, 2, 4, DELTA_INF), policies=("isjl",), robust=True,
                note="n=6 at t=0; prompt U[1,4]; output U[1,8]; slack U{0..3}"),
    8: Workload(8, "online-robust", 10_000, 1_000, 8000, B=(256,), kv_caps=(200_000,),
                deltas=(16, 64, 256, 1024, DELTA_INF), online=True, robust=True,
                note="workload 3's distributions; slack = rint(output * U[0, 0.5])"),
}


def chunk_instances(n_per_instance: int) -> int:
    """Instances per independently seeded chunk (a power of two, ~2**20 requests)."""
    target = max(1, (1 << 20) // max(1, n_per_instance))
    return 1 << int(math.floor(math.log2(target)))


def _poisson_arrivals(rng, shape, mean_gap):
    gaps = rng.exponential(mean_gap, size=shape)
    return np.floor(np.cumsum(gaps, axis=1)).astype(np.int32)


def _lognormal_int(rng, shape, median, sigma, lo, hi):
    x = np.rint(rng.lognormal(mean=math.log(median), sigma=sigma, size=shape))
    return np.clip(x, lo, hi).astype(np.int32)


def _draw_chunk(wl: Workload, chunk: int, rows: int, replica: int = 0):
    key = [wl.seed, chunk] + ([replica] if replica else [])
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(key)))
    n = wl.n_per_instance
    shape = (rows, n)
    if wl.wid == 1:
        arrival = np.zeros(shape, np.int32)
        prompt = rng.integers(1, 33, size=shape, dtype=np.int32)
        short = rng.random(shape) < 0.7
        out_s = rng.integers(1, 17, size=shape, dtype=np.int32)
        out_l = rng.integers(64, 257, size=shape, dtype=np.int32)
        output = np.where(short, out_s, out_l).astype(np.int32)
    elif wl.wid == 2:
        arrival = np.zeros(shape, np.int32)
        prompt = rng.integers(1, 5, size=shape, dtype=np.int32)
        output = rng.integers(1, 9, size=shape, dtype=np.int32)
    elif wl.wid == 3:
        arrival = _poisson_arrivals(rng, shape, 2.0)
        prompt = _lognormal_int(rng, shape, 512, 1.0, 16, 4096)
        output = _lognormal_int(rng, shape, 256, 1.2, 1, 2048)
    elif wl.wid == 4:
        arrival = np.zeros(shape, np.int32)
        prompt = rng.integers(16, 1025, size=shape, dtype=np.int32)
        x = np.floor(8.0 * (1.0 + rng.pareto(1.5, size=shape)))
        output = np.clip(x, 8, 8192).astype(np.int32)
    elif wl.wid == 5:
        arrival = _poisson_arrivals(rng, shape, 0.05)
        prompt = _lognormal_int(rng, shape, 1024, 1.0, 16, 32768)
        output = _lognormal_int(rng, shape, 512, 1.3, 1, 16384)
    elif wl.wid == 6:
        offered = rng.integers(1, 1001, size=shape)
        u = rng.random(shape)
        bucket = (offered + 99) // 100
        keep = u < np.maximum(0.0, 1.0 - offered / ((2 * bucket - 1) * 100.0))
        count = keep.sum(axis=1).astype(np.int32)
        arrival = np.zeros(shape, np.int32)
        prompt = np.zeros(shape, np.int32)
        output = np.zeros(shape, np.int32)
        for r in range(rows):                       # accepted requests first, in offer order
            acc = offered[r][keep[r]]
            output[r, :acc.size] = acc
        return arrival, prompt, output, count, None
    elif wl.wid == 7:
        arrival = np.zeros(shape, np.int32)
        prompt = rng.integers(1, 5, size=shape, dtype=np.int32)
        output = rng.integers(1, 9, size=shape, dtype=np.int32)
        slack = rng.integers(0, 4, size=shape, dtype=np.int32)
        return arrival, prompt, output, None, slack
    elif wl.wid == 8:
        arrival = _poisson_arrivals(rng, shape, 2.0)
        prompt = _lognormal_int(rng, shape, 512, 1.0, 16, 4096)
        output = _lognormal_int(rng, shape, 256, 1.2, 1, 2048)
        slack = np.rint(output * rng.uniform(0.0, 0.5, size=shape)).astype(np.int32)
        return arrival, prompt, output, None, slack
    else:  # pragma: no cover
        raise ValueError(f"unknown workload {wl.wid}")
    return arrival, prompt, output, None, None


def generate(wid: int, instances=None, replica: int = 0, with_counts: bool = False, with_slack: bool = False):
    """Return (arrival, prompt, output), each int32 of shape (len(instances), n).

    ``instances`` is None (all instances), an int m (the first m) or an
    iterable of instance ids.  Instance i is identical whichever way it is
    requested.  ``replica`` r > 0 draws an independent set of the same shape
    (seed sequence [seed, chunk, r]); multi-GPU runs give rank r replica r.
    ``with_counts`` appends the per-instance request counts (all n except for
    ragged workloads, whose instance i uses its first counts[i] slots);
    ``with_slack`` then appends the upper-bound slack array (zeros unless the
    workload is robust).
    """
    wl = WORKLOADS[wid]
    if instances is None:
        ids = np.arange(wl.n_instances)
    elif isinstance(instances, (int, np.integer)):
        ids = np.arange(min(int(instances), wl.n_instances))
    else:
        ids = np.asarray(list(instances), dtype=np.int64)
    if ids.size and (ids.min() < 0 or ids.max() >= wl.n_instances):
        raise IndexError("instance id out of range")
    per = chunk_instances(wl.n_per_instance)
    n = wl.n_per_instance
    out = [np.empty((ids.size, n), np.int32) for _ in range(3)]
    cnt = np.empty(ids.size, np.int32)
    slk = np.zeros((ids.size, n), np.int32)
    chunks = ids // per
    for c in np.unique(chunks):
        sel = np.nonzero(chunks == c)[0]
        # always draw the whole chunk: later arrays depend on how many values
        # the earlier draws consumed
        rows = min(per, wl.n_instances - int(c) * per)
        arrs = _draw_chunk(wl, int(c), rows, replica)
        for k in range(3):
            out[k][sel] = arrs[k][ids[sel] % per]
        cnt[sel] = arrs[3][ids[sel] % per] if arrs[3] is not None else n
        if arrs[4] is not None:
            slk[sel] = arrs[4][ids[sel] % per]
    res = tuple(out)
    if with_counts:
        res = res + (cnt,)
    if with_slack:
        res = res + (slk,)
    return res


def custom(arrival, prompt, output):
    """Validate and pack caller-made instances into contiguous int32 arrays."""
    a = np.ascontiguousarray(np.atleast_2d(np.asarray(arrival, dtype=np.int32)))
    p = np.ascontiguousarray(np.atleast_2d(np.asarray(prompt, dtype=np.int32)))
    o = np.ascontiguousarray(np.atleast_2d(np.asarray(output, dtype=np.int32)))
    if not (a.shape == p.shape == o.shape):
        raise ValueError("arrival/prompt/output shapes differ")
    return a, p, o
