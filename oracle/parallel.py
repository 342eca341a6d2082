"""The oracle over many instances on every host core (test infrastructure only).

Only tests and the benchmark's CPU legs may use this module.  Work is split
into blocks of consecutive instances, one task per block, on a process pool
made with the "spawn" start method: the children are fresh interpreters, so
the pool is safe to create after the parent has used a GPU.
"""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np


def _block(args):
    policy, B, delta, kv, a, p, o, counts, slack, per_request = args
    from oracle import oracle as O
    return O.run(policy, B, delta, kv, a, p, o, per_request=per_request, counts=counts, slack=slack)


def make_pool(processes=None):
    return mp.get_context("spawn").Pool(processes or os.cpu_count() or 1)


def run(pool, policy, B, delta, kv, arrival, prompt, output, per_request=False, counts=None, slack=None,
        block=None):
    """oracle.run over all rows of the (n_instances, n) arrays, split across
    the pool; returns (records, start, completion) like oracle.run."""
    n_inst = len(arrival)
    if block is None:
        block = max(1, -(-n_inst // (4 * pool._processes)))
    jobs = []
    for s in range(0, n_inst, block):
        e = min(n_inst, s + block)
        jobs.append((policy, B, delta, kv, arrival[s:e], prompt[s:e], output[s:e],
                     None if counts is None else counts[s:e], None if slack is None else slack[s:e],
                     per_request))
    res = pool.map(_block, jobs)
    rec = np.concatenate([r[0] for r in res])
    if not per_request:
        return rec, None, None
    return rec, np.concatenate([r[1] for r in res]), np.concatenate([r[2] for r in res])
