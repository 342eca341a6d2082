"""ctypes front end of the CPU oracle (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this module.  It loads ``oracle/_build/liboracle.so`` (built by
``oracle/build.py``) and exposes:

  run(policy, B, delta, kv_cap, arrival, prompt, output, ...) -> (records, start, completion)
  opt_makespan(arrival, o, B, delta, kv_cap) -> optimal makespan (tiny instances)

``policy`` is "fcfs", "ljf" or "isjl".  Arrays are int32 of shape
(n_instances, n) or (n,).  ``delta``/``kv_cap`` of INT32_MAX mean "no limit".
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

INT32_MAX = 2**31 - 1
POLICIES = {"fcfs": 0, "ljf": 1, "isjl": 2, "sjf": 3, "isjl_beta": 4}
STATUS = {0: "ok", 1: "invalid_arg", 2: "infeasible", 3: "oom", 5: "step_limit"}

RECORD_FIELDS_I64 = ["T_make", "T_busy", "O", "Q", "W", "E", "token_adv",
                     "sum_completion", "sum_latency", "sum_extent", "max_extent",
                     "violations", "kv_violations", "peak_kv", "peak_batch", "status"]
RECORD_FIELDS_F64 = ["c_T", "tau_Q", "tau_E", "cost", "revenue", "profit", "throughput", "ael"]
RECORD_DTYPE = np.dtype([(f, np.int64) for f in RECORD_FIELDS_I64] +
                        [(f, np.float64) for f in RECORD_FIELDS_F64])

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        p32 = ctypes.POINTER(ctypes.c_int32)
        L.oracle_run_batch.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                       ctypes.c_int, ctypes.c_int, p32, p32, p32, p32,
                                       ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                       ctypes.c_int64, p32, p32, ctypes.c_void_p]
        L.oracle_run_batch.restype = ctypes.c_int
        L.oracle_run_batch_v.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                         ctypes.c_int, ctypes.c_int, p32, p32, p32, p32,
                                         ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                         ctypes.c_int64, ctypes.c_int, p32, p32, ctypes.c_void_p]
        L.oracle_run_batch_v.restype = ctypes.c_int
        L.oracle_record_size.restype = ctypes.c_int
        L.oracle_beta.argtypes = [ctypes.c_int64]
        L.oracle_beta.restype = ctypes.c_int64
        L.oracle_opt_makespan.argtypes = [ctypes.c_int, p32, p32, ctypes.c_int, ctypes.c_int64,
                                          ctypes.c_int64, ctypes.c_int64]
        L.oracle_opt_makespan.restype = ctypes.c_int64
        if L.oracle_record_size() != RECORD_DTYPE.itemsize:
            raise RuntimeError("oracle record layout mismatch")
        _lib = L
    return _lib


def _i32(x):
    return np.ascontiguousarray(np.asarray(x, dtype=np.int32))


def _ptr(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


# ISJL reading variants (the reading study only; 0 = the specified readings)
VARIANTS = {"no_wait_o1": 1, "d1_last": 2, "p2_reserved": 4, "rebuild_reopen": 8, "literal_long": 16,
            "short_packs": 32, "cancel": 64, "waiver": 128, "ungated_plan": 256}


def run(policy, B, delta, kv_cap, arrival, prompt, output, c=0.0005, tau=1e-6, p0=0.002,
        max_steps=0, per_request=True, counts=None, slack=None, variant=0):
    """Simulate every instance (row) under one policy and budget.

    Returns (records, start, completion); records is a structured array with
    one entry per instance (fields RECORD_DTYPE), start/completion are int32
    arrays shaped like ``arrival`` (None when per_request is False).
    ``counts`` (optional, one per row) limits instance i to its first
    counts[i] requests (ragged batches); the rest stay -1.  ``slack`` (optional,
    shaped like ``arrival``) is the upper-bound slack e_i = u_i - o_i: policies
    plan with u_i and requests finish after o_i tokens (Robust-ISJL).
    ``variant`` ORs VARIANTS flags: alternative readings of Algorithm 2, used
    only by the reading study; 0 is the simulator's specification.
    """
    if counts is not None:
        a, p, o = (np.atleast_2d(_i32(x)) for x in (arrival, prompt, output))
        e = np.atleast_2d(_i32(slack)) if slack is not None else None
        recs, sts, cos = [], [], []
        for i, m in enumerate(np.asarray(counts)):
            m = int(m)
            if m < 0 or m > a.shape[1]:            # a count outside 0..n: invalid instance
                r = np.zeros(1, RECORD_DTYPE)
                r["status"] = 1
                recs.append(r)
                if per_request:
                    sts.append(np.full((1, a.shape[1]), -1, np.int32))
                    cos.append(np.full((1, a.shape[1]), -1, np.int32))
                continue
            r, st, co = run(policy, B, delta, kv_cap, a[i:i + 1, :m], p[i:i + 1, :m], o[i:i + 1, :m], c, tau, p0,
                            max_steps, per_request, slack=e[i:i + 1, :m] if e is not None else None,
                            variant=variant)
            recs.append(r)
            if per_request:
                row = np.full((1, a.shape[1]), -1, np.int32)
                rc = row.copy()
                row[0, :m] = st[0, :m] if m else row[0, :0]
                rc[0, :m] = co[0, :m] if m else rc[0, :0]
                sts.append(row)
                cos.append(rc)
        rec = np.concatenate(recs)
        return rec, (np.concatenate(sts) if per_request else None), (np.concatenate(cos) if per_request else None)
    a, p, o = _i32(arrival), _i32(prompt), _i32(output)
    e = _i32(slack) if slack is not None else None
    squeeze = a.ndim == 1
    if squeeze:
        a, p, o = a[None], p[None], o[None]
        e = e[None] if e is not None else None
    n_inst, n = a.shape
    rec = np.zeros(n_inst, RECORD_DTYPE)
    st = np.full((n_inst, n), -1, np.int32) if per_request else None
    co = np.full((n_inst, n), -1, np.int32) if per_request else None
    lib().oracle_run_batch_v(POLICIES[policy], int(B), int(delta), int(kv_cap), n_inst, n,
                             _ptr(a), _ptr(p), _ptr(o), _ptr(e) if e is not None else None,
                             float(c), float(tau), float(p0), int(max_steps), int(variant),
                             _ptr(st) if per_request else None, _ptr(co) if per_request else None,
                             rec.ctypes.data)
    if squeeze:
        rec = rec[0]
        st = st[0] if per_request else None
        co = co[0] if per_request else None
    return rec, st, co


def beta(alpha):
    """floor((sqrt(17) - 1) / 4 * alpha), Algorithm "ISJL"'s beta, exact."""
    return int(lib().oracle_beta(int(alpha)))


def opt_makespan(arrival, o, B, delta, kv_cap=INT32_MAX, max_T=100_000):
    """Exact optimal makespan of one tiny instance (n <= 9, o_i <= 62)."""
    a, oo = _i32(arrival), _i32(o)
    return int(lib().oracle_opt_makespan(len(oo), _ptr(a), _ptr(oo), int(B), int(delta),
                                         int(kv_cap), int(max_T)))
