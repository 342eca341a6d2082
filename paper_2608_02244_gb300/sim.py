"""Python binding of the C-ABI simulator library (argument marshalling only).

Every function here forwards to the entry point of the same name declared in
``include/isjl_sim.h``; all simulation work runs in the library's CUDA
kernels.  PyTorch supplies device memory and streams.  Importing this module
fails loudly if the shared library has not been built (``build()`` in
``__graft_entry__`` or ``python -m paper_2608_02244_gb300.build``): there is
no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libisjl_sim.so")

ISJL_OK, ISJL_ERR_INVALID_ARG, ISJL_ERR_INFEASIBLE, ISJL_ERR_OOM = 0, 1, 2, 3
ISJL_ERR_CUDA, ISJL_ERR_STEP_LIMIT, ISJL_ERR_NOT_READY, ISJL_ERR_INTERNAL = 4, 5, 6, 7
POLICY = {"fcfs": 0, "ljf": 1, "isjl": 2, "sjf": 3, "isjl_beta": 4}
DELTA_INF = 2**31 - 1
KV_INF = 2**31 - 1
MAX_B, MAX_LEN, MAX_RUNS = 512, 65535, 32
FLAG_STEP_KERNEL, FLAG_EPOCH_KERNEL, FLAG_TIMING = 0, 1, 2

_I64 = ["T_make", "T_busy", "O", "Q", "W", "E", "token_adv", "sum_completion", "sum_latency",
        "sum_extent", "max_extent", "violations", "kv_violations", "peak_kv", "peak_batch", "status"]
_F64 = ["c_T", "tau_Q", "tau_E", "cost", "revenue", "profit", "throughput", "ael"]
RECORD_DTYPE = np.dtype([(f, np.int64) for f in _I64] + [(f, np.float64) for f in _F64])


class isjl_config(ctypes.Structure):
    _fields_ = [("n_instances", ctypes.c_int64), ("n_per_instance", ctypes.c_int32), ("B", ctypes.c_int32),
                ("c", ctypes.c_double), ("tau", ctypes.c_double), ("p0", ctypes.c_double),
                ("max_steps", ctypes.c_int64), ("flags", ctypes.c_uint32)]


class isjl_instances(ctypes.Structure):
    _fields_ = [("arrival", ctypes.c_void_p), ("prompt", ctypes.c_void_p), ("output", ctypes.c_void_p),
                ("count", ctypes.c_void_p), ("slack", ctypes.c_void_p)]


class isjl_outputs(ctypes.Structure):
    _fields_ = [("records", ctypes.c_void_p), ("start", ctypes.c_void_p), ("completion", ctypes.c_void_p)]


class isjl_record(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in _I64] + [(f, ctypes.c_double) for f in _F64]


class isjl_summary(ctypes.Structure):
    _fields_ = ([("policy", ctypes.c_int32), ("delta", ctypes.c_int32), ("kv_cap", ctypes.c_int32),
                 ("status", ctypes.c_int32), ("n_instances", ctypes.c_int64), ("n_ok", ctypes.c_int64)] +
                [(f, ctypes.c_int64) for f in ["T_make", "T_busy", "O", "Q", "W", "E", "token_adv",
                                               "sum_completion", "sum_latency", "sum_extent", "max_extent",
                                               "violations", "kv_violations"]] +
                [(f, ctypes.c_double) for f in ["c_T", "tau_Q", "tau_E", "cost", "revenue", "profit"]])


assert ctypes.sizeof(isjl_record) == RECORD_DTYPE.itemsize == 192

EXPORTS = ["isjl_sim_create", "isjl_sim_destroy", "isjl_sim_run", "isjl_sim_run_sweep",
           "isjl_sim_run_sweep_host", "isjl_sim_metrics", "isjl_sim_last_launches", "isjl_sim_kernel_times",
           "isjl_sim_run_sweep_noalloc", "isjl_probe_int_rate", "isjl_status_string"]

_lib = None


def lib():
    """Load the shared library (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"CUDA simulator library missing: {LIB_PATH} (run the build step first)")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, p32 = ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32)
        L.isjl_sim_create.argtypes = [ctypes.POINTER(isjl_config), ctypes.POINTER(vp)]
        L.isjl_sim_create.restype = ctypes.c_int
        L.isjl_sim_destroy.argtypes = [vp]
        L.isjl_sim_destroy.restype = None
        L.isjl_sim_run.argtypes = [vp, ctypes.c_int, i32, i32, ctypes.POINTER(isjl_instances),
                                   ctypes.POINTER(isjl_outputs), vp]
        L.isjl_sim_run.restype = ctypes.c_int
        L.isjl_sim_run_sweep.argtypes = [vp, i32, p32, p32, i32, ctypes.POINTER(isjl_instances),
                                         ctypes.POINTER(isjl_outputs), vp]
        L.isjl_sim_run_sweep.restype = ctypes.c_int
        L.isjl_sim_run_sweep_host.argtypes = [vp, i32, p32, p32, i32, vp, vp, vp, vp, vp, vp, vp]
        L.isjl_sim_run_sweep_host.restype = ctypes.c_int
        L.isjl_sim_metrics.argtypes = [vp, ctypes.POINTER(isjl_summary), i32]
        L.isjl_sim_metrics.restype = ctypes.c_int
        L.isjl_sim_last_launches.argtypes = [vp]
        L.isjl_sim_last_launches.restype = i32
        L.isjl_sim_kernel_times.argtypes = [vp, ctypes.POINTER(ctypes.c_float), i32]
        L.isjl_sim_kernel_times.restype = i32
        L.isjl_sim_run_sweep_noalloc.argtypes = [ctypes.POINTER(isjl_config), i32, p32, p32, i32,
                                                 ctypes.POINTER(isjl_instances), ctypes.POINTER(isjl_outputs), vp]
        L.isjl_sim_run_sweep_noalloc.restype = ctypes.c_int
        L.isjl_probe_int_rate.argtypes = [i32, i32, vp, ctypes.POINTER(ctypes.c_double),
                                          ctypes.POINTER(ctypes.c_float)]
        L.isjl_probe_int_rate.restype = ctypes.c_int
        L.isjl_status_string.argtypes = [ctypes.c_int]
        L.isjl_status_string.restype = ctypes.c_char_p
        _lib = L
    return _lib


class IsjlError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {isjl_status_string(status)} ({status})")


def isjl_status_string(status: int) -> str:
    return lib().isjl_status_string(int(status)).decode()


def _check(st, where):
    if st != ISJL_OK:
        raise IsjlError(st, where)


def _i32_array(vals):
    a = (ctypes.c_int32 * len(vals))(*[int(v) for v in vals])
    return a


def _policy_code(p):
    return POLICY[p] if isinstance(p, str) else int(p)


# ---- thin wrappers with the C names ----------------------------------------
def isjl_probe_int_rate(kind, iters, stream=None):
    """(int32 lane-instructions executed, milliseconds) of one probe launch;
    kind 0 = adds, 1 = min / max."""
    n = ctypes.c_double()
    ms = ctypes.c_float()
    _check(lib().isjl_probe_int_rate(int(kind), int(iters), _stream_ptr(stream), ctypes.byref(n), ctypes.byref(ms)),
           "isjl_probe_int_rate")
    return n.value, ms.value


def isjl_sim_create(n_instances, n_per_instance, B, c=0.0005, tau=1e-6, p0=0.002, max_steps=0,
                    flags=FLAG_STEP_KERNEL):
    cfg = isjl_config(int(n_instances), int(n_per_instance), int(B), float(c), float(tau), float(p0),
                      int(max_steps), int(flags))
    h = ctypes.c_void_p()
    _check(lib().isjl_sim_create(ctypes.byref(cfg), ctypes.byref(h)), "isjl_sim_create")
    return h


def isjl_sim_destroy(handle):
    if handle:
        lib().isjl_sim_destroy(handle)


def _stream_ptr(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(stream.cuda_stream))


def _instances(arrival, prompt, output, count, slack=None):
    return isjl_instances(arrival.data_ptr(), prompt.data_ptr(), output.data_ptr(),
                          count.data_ptr() if count is not None else None,
                          slack.data_ptr() if slack is not None else None)


def isjl_sim_run(handle, policy, delta, kv_cap, arrival, prompt, output, records, start=None,
                 completion=None, stream=None, count=None):
    ins = _instances(arrival, prompt, output, count)
    outs = isjl_outputs(records.data_ptr(), start.data_ptr() if start is not None else None,
                        completion.data_ptr() if completion is not None else None)
    return lib().isjl_sim_run(handle, _policy_code(policy), int(delta), int(kv_cap), ctypes.byref(ins),
                              ctypes.byref(outs), _stream_ptr(stream))


def isjl_sim_run_sweep(handle, policies, deltas, kv_cap, arrival, prompt, output, records, start=None,
                       completion=None, stream=None, count=None, slack=None):
    pol = _i32_array([_policy_code(p) for p in policies])
    dl = _i32_array(deltas)
    ins = _instances(arrival, prompt, output, count, slack)
    outs = isjl_outputs(records.data_ptr(), start.data_ptr() if start is not None else None,
                        completion.data_ptr() if completion is not None else None)
    return lib().isjl_sim_run_sweep(handle, len(pol), pol, dl, int(kv_cap), ctypes.byref(ins),
                                    ctypes.byref(outs), _stream_ptr(stream))


def isjl_sim_run_sweep_host(handle, policies, deltas, kv_cap, h_arrival, h_prompt, h_output, h_records,
                            stream=None, h_count=None, h_slack=None):
    """Host-memory sweep: h_* are pinned (or pageable) torch CPU int32 tensors
    (h_count / h_slack optional), h_records a CPU uint8 tensor of
    n_runs * n_instances * 192 bytes."""
    pol = _i32_array([_policy_code(p) for p in policies])
    dl = _i32_array(deltas)
    return lib().isjl_sim_run_sweep_host(handle, len(pol), pol, dl, int(kv_cap), h_arrival.data_ptr(),
                                         h_prompt.data_ptr(), h_output.data_ptr(),
                                         h_count.data_ptr() if h_count is not None else None,
                                         h_slack.data_ptr() if h_slack is not None else None,
                                         h_records.data_ptr(), _stream_ptr(stream))


def isjl_sim_run_sweep_noalloc(n_instances, n_per_instance, B, policies, deltas, kv_cap, arrival, prompt,
                               output, records, start=None, completion=None, c=0.0005, tau=1e-6, p0=0.002,
                               max_steps=0, flags=FLAG_STEP_KERNEL, stream=None, count=None, slack=None):
    """Allocation-free sweep for callers that cannot allocate device memory at the
    point of use (allocator-owned pools, fixed budgets, no-sync sections): the
    library's workspace is a fixed device array shared by all calls, so calls
    must not overlap on the GPU.  Device int32 tensors in, device buffers out;
    returns the status code (no exception, no summaries)."""
    cfg = isjl_config(int(n_instances), int(n_per_instance), int(B), float(c), float(tau), float(p0),
                      int(max_steps), int(flags))
    pol = _i32_array([_policy_code(p) for p in policies])
    dl = _i32_array(deltas)
    ins = _instances(arrival, prompt, output, count, slack)
    outs = isjl_outputs(records.data_ptr(), start.data_ptr() if start is not None else None,
                        completion.data_ptr() if completion is not None else None)
    return lib().isjl_sim_run_sweep_noalloc(ctypes.byref(cfg), len(pol), pol, dl, int(kv_cap), ctypes.byref(ins),
                                            ctypes.byref(outs), _stream_ptr(stream))


def isjl_sim_metrics(handle, max_runs=MAX_RUNS):
    arr = (isjl_summary * max_runs)()
    st = lib().isjl_sim_metrics(handle, arr, max_runs)
    return st, arr


def isjl_sim_last_launches(handle) -> int:
    return int(lib().isjl_sim_last_launches(handle))


def isjl_sim_kernel_times(handle):
    """Durations (ms) of derive, sort, simulate, summarize of the last call."""
    arr = (ctypes.c_float * 4)()
    k = lib().isjl_sim_kernel_times(handle, arr, 4)
    if k < 0:
        raise IsjlError(ISJL_ERR_CUDA, "isjl_sim_kernel_times")
    return [float(arr[i]) for i in range(k)]


# ---- convenience layer ------------------------------------------------------
def summary_to_dict(s: isjl_summary) -> dict:
    return {f: getattr(s, f) for f, _ in isjl_summary._fields_}


def records_to_numpy(records_tensor, n_runs, n_inst):
    """View a uint8 records tensor (device or host) as (n_runs, n_inst) RECORD_DTYPE."""
    host = records_tensor.detach().cpu().numpy()
    return host.view(RECORD_DTYPE).reshape(n_runs, n_inst)


class Simulator:
    """Owns a library handle plus torch output buffers for one instance shape."""

    def __init__(self, n_instances, n_per_instance, B, c=0.0005, tau=1e-6, p0=0.002, max_steps=0,
                 epoch=False, timing=False):
        import torch
        self.torch = torch
        self.n_inst, self.n, self.B = int(n_instances), int(n_per_instance), int(B)
        flags = (FLAG_EPOCH_KERNEL if epoch else FLAG_STEP_KERNEL) | (FLAG_TIMING if timing else 0)
        self.handle = isjl_sim_create(n_instances, n_per_instance, B, c, tau, p0, max_steps, flags)
        self._records = None
        self._per_req = None

    def close(self):
        if self.handle:
            isjl_sim_destroy(self.handle)
            self.handle = None

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass

    def buffers(self, n_runs, per_request):
        torch = self.torch
        need = n_runs * self.n_inst * RECORD_DTYPE.itemsize
        if self._records is None or self._records.numel() < need:
            self._records = torch.empty(need, dtype=torch.uint8, device="cuda")
        rec = self._records[:need]
        st = co = None
        if per_request:
            npr = n_runs * self.n_inst * self.n
            if self._per_req is None or self._per_req[0].numel() < npr:
                self._per_req = (torch.empty(npr, dtype=torch.int32, device="cuda"),
                                 torch.empty(npr, dtype=torch.int32, device="cuda"))
            st, co = self._per_req[0][:npr], self._per_req[1][:npr]
        return rec, st, co

    def sweep_async(self, arrival, prompt, output, policies, deltas, kv_cap, per_request=False, stream=None,
                    counts=None, slack=None):
        """Launch a sweep on device-resident int32 tensors; returns output tensors."""
        rec, st, co = self.buffers(len(policies), per_request)
        if per_request:
            st.fill_(-1)
            co.fill_(-1)
        _check(isjl_sim_run_sweep(self.handle, policies, deltas, kv_cap, arrival, prompt, output, rec, st, co,
                                  stream, counts, slack), "isjl_sim_run_sweep")
        return rec, st, co

    def sweep(self, arrival, prompt, output, policies, deltas, kv_cap, per_request=False, stream=None,
              counts=None, slack=None):
        """Run a sweep and return numpy results: records (n_runs, n_inst), start and
        completion (n_runs, n_inst, n) or None, per-run summaries, device status."""
        torch = self.torch

        def dev(x):
            t = torch.as_tensor(np.ascontiguousarray(x, dtype=np.int32)) if not torch.is_tensor(x) else x
            return t.to(device="cuda", dtype=torch.int32).contiguous()

        a, p, o = dev(arrival), dev(prompt), dev(output)
        cnt = dev(counts) if counts is not None else None
        sl = dev(slack) if slack is not None else None
        rec, st, co = self.sweep_async(a, p, o, policies, deltas, kv_cap, per_request, stream, cnt, sl)
        status, summ = isjl_sim_metrics(self.handle)
        R = len(policies)
        out = {
            "records": records_to_numpy(rec, R, self.n_inst),
            "summaries": [summary_to_dict(summ[i]) for i in range(R)],
            "status": status,
            "launches": isjl_sim_last_launches(self.handle),
        }
        if per_request:
            out["start"] = st.cpu().numpy().reshape(R, self.n_inst, self.n)
            out["completion"] = co.cpu().numpy().reshape(R, self.n_inst, self.n)
        return out
