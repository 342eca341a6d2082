#!/usr/bin/env python
"""Benchmark: simulated batch-steps per second of the online delta-sweep.

One step = one sweep of the whole hot path (derive, sort, simulate,
summarize) over the online delta-sweep workload: 10,000 instances x 1,000
requests (Poisson arrivals, mean gap 2 steps; prompt lognormal(ln 512, 1)
clipped [16, 4096]; output lognormal(ln 256, 1.2) clipped [1, 2048]), KV cap
200,000 tokens, B = 256 batch slots, runs FCFS, LJF and ISJL at
delta in {16, 64, 256, 1024, inf} (7 runs per instance), per-request start and
completion steps written out.  A batch-step is a simulated step whose batch
is nonempty; value = sum over (instance, run) of T_busy per second.
--workload picks another workload's run grid (GRIDS below) for the same
measurement; the default line is the online delta-sweep.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--kernel step|epoch] [--workload 3|4|5|6|8]
  python bench.py --impl reference ...     (the CPU oracle on host cores)

Multi-GPU (torchrun): rank r simulates its own replica of the workload
(independent instances, weak scaling, no collective on the data path); the
timing is the max over ranks.  Prints one JSON line on rank 0.
"""
from __future__ import annotations

import argparse
import json
import multiprocessing as mp
import os
import platform
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_02244_gb300 import workloads as W  # noqa: E402

METRIC = "simulated batch-steps/sec on 1 GB300 (ISJL Δ-sweep); % of HBM/int roofline"
UNIT = "batch-steps/s"
INF = W.DELTA_INF
DEFAULT_WID = 3
# per workload: (policies, fairness budgets, oracle instances per host core for
# the CPU baseline sample: one to two seconds of oracle work per core)
GRIDS = {
    1: (["fcfs", "ljf", "isjl"], [0, 0, 32], 1),
    2: (["isjl"] * 5, [0, 1, 2, 4, INF], 256),
    3: (["fcfs", "ljf", "isjl", "isjl", "isjl", "isjl", "isjl"], [0, 0, 16, 64, 256, 1024, INF], 40),
    4: (["fcfs", "ljf", "isjl", "isjl", "isjl"], [0, 0, 32, 128, 512], 400),
    5: (["fcfs", "ljf", "isjl"], [0, 0, 256], 1),
    6: (["fcfs", "ljf"] + ["isjl"] * 7, [0, 0, 50, 100, 150, 250, 300, 400, 500], 400),
    8: (["fcfs", "ljf", "isjl", "isjl", "isjl", "isjl", "isjl"], [0, 0, 16, 64, 256, 1024, INF], 40),
}
# nominal int32 lanes per SM on GB300 (4 SM sub-partitions x 32 lanes), for context
ALU_LANES_PER_SM = 128
# algorithmic integer work of the per-step kernel: per token-advance
# (r = a + 1, store, max, min, add/compare) and per batch-step (W, E, extent,
# violation, T_busy, token counter)
OPS_PER_TOKEN_ADVANCE = 5
OPS_PER_BATCH_STEP = 6
# algorithmic integer work of the event-driven kernel: per request start or
# completion (KV reservation, earliest completion / start range, counter,
# output store, queue bit) and per epoch, a step at which a request starts or
# completes (the closed-form W, E, extent, max extent, violations, T_busy and
# token terms of the interval that follows)
OPS_PER_REQUEST_EVENT = 5
OPS_PER_EPOCH = 14
# probe launches for the measured integer rates: iterations per thread (about
# 30-60 ms per launch on GB300) and launches per kind (the fastest is kept)
PROBE_ITERS = 20_000
PROBE_LAUNCHES = 3
# DRAM bytes (read + write) per launch of the step simulation kernel on the full
# workload: 742.6 MB measured by ncu on the first 4,096 instances, scaled by
# 10,000 / 4,096 (profiles/sim_kernel_step_online_delta_sweep_4096.md)
SIM_DRAM_BYTES_PER_LAUNCH = 742.6e6 * 10_000 / 4_096
# issue-slot and ALU-pipe utilisation of the same capture (smsp__issue_active and
# sm__inst_executed_pipe_alu, percent of peak while active), reported beside the roofline
SIM_NCU_ISSUE_ACTIVE = 0.750
SIM_NCU_ALU_PIPE = 0.681


def workload_config(kernel, wl, n_inst, policies, deltas, flush):
    kv = "none" if wl.kv_caps[0] == W.KV_INF else wl.kv_caps[0]
    return {
        "workload": f"{wl.name}: {n_inst} instances x {wl.n_per_instance} requests, {wl.note}",
        "B": wl.B[0], "kv_cap": kv, "policies": policies,
        "deltas": ["inf" if d == INF else d for d in deltas],
        "runs_per_instance": len(policies), "per_request_outputs": True,
        "kernel": kernel, "l2": flush,
    }


# ---------------------------------------------------------------- clocks ----
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons while timing."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid=None):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if uuid:
            cmd += ["-i", uuid]
        try:
            self.p = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------ measured peaks ----
def probe_peaks(sim, stream):
    """Measured int32 issue rates (Tops/s): adds and min / max, best of
    PROBE_LAUNCHES launches each (isjl_probe_int_rate)."""
    out = {}
    for kind, name in ((0, "add"), (1, "minmax")):
        best = 0.0
        for _ in range(PROBE_LAUNCHES):
            n, ms = sim.isjl_probe_int_rate(kind, PROBE_ITERS, stream)
            best = max(best, n / (ms / 1e3) / 1e12)
        out[name] = best
    return out


def epoch_count(start, completion):
    """Steps at which some request starts or completes, summed over (run,
    instance): the epochs the event-driven kernel closes in closed form."""
    runs = start.shape[0]
    total = 0
    for r in range(runs):
        ev = np.concatenate([start[r], completion[r]], axis=1)
        ev = np.sort(ev, axis=1)
        valid = ev >= 0
        new = np.ones_like(valid)
        new[:, 1:] = ev[:, 1:] != ev[:, :-1]
        total += int((valid & new).sum())
    return total


# ------------------------------------------------------------ CPU oracle ----
def _oracle_chunk(args):
    """Worker: run the oracle on a block of instances; returns (sum T_busy, sum token_adv)."""
    a, p, o, cnt, slack, B, kv, policies, deltas = args
    sys.path.insert(0, ROOT)
    from oracle import oracle as O
    tb = tok = 0
    for pol, d in zip(policies, deltas):
        rec, _, _ = O.run(pol, B, d, kv, a, p, o, per_request=False, counts=cnt, slack=slack)
        tb += int(rec["T_busy"].sum())
        tok += int(rec["token_adv"].sum())
    return tb, tok


def oracle_timed(inputs, B, kv, policies, deltas, cores, pool):
    """Oracle over `inputs` split into one block per core; (sum T_busy, sum
    token advances, wall seconds, blocks)."""
    a, p, o, cnt, slack = inputs
    chunks = [x for x in np.array_split(np.arange(len(a)), cores) if len(x)]
    jobs = [(a[c], p[c], o[c], None if cnt is None else cnt[c], None if slack is None else slack[c],
             B, kv, policies, deltas) for c in chunks]
    t = time.perf_counter()
    res = pool.map(_oracle_chunk, jobs)
    dt = time.perf_counter() - t
    return sum(r[0] for r in res), sum(r[1] for r in res), dt, len(jobs)


def host_inputs(wid, count, replica=0):
    """(arrival, prompt, output, counts or None, slack or None) of the first
    `count` instances; counts only for ragged workloads, slack only for robust."""
    wl = W.WORKLOADS[wid]
    a, p, o, cnt, slack = W.generate(wid, count, replica=replica, with_counts=True, with_slack=True)
    return a, p, o, (cnt if wl.ragged else None), (slack if wl.robust else None)


def cpu_model():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.processor() or platform.machine()


# --------------------------------------------------------------- dist -------
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def combine_ranks(t_ms, units, e2e_ms, dist=None, device="cpu"):
    """Whole-job figures: the max over ranks of the timed milliseconds (and of
    the e2e milliseconds) and the sum over ranks of the units processed."""
    if dist is None:
        return t_ms, units, e2e_ms
    import torch
    t = torch.tensor([t_ms, e2e_ms], dtype=torch.float64, device=device)
    u = torch.tensor([units], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t[0]), float(u[0]), float(t[1])


def reference_arm(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    wl = W.WORKLOADS[args.workload]
    policies, deltas, per_core = GRIDS[args.workload]
    per_core = max(1, per_core * 3 // 10)
    cores = args.oracle_cores or os.cpu_count() or 1
    inputs = host_inputs(args.workload, cores * per_core)
    ctx = mp.get_context("spawn")
    with ctx.Pool(cores) as pool:
        for _ in range(args.warmup):
            oracle_timed(inputs, wl.B[0], wl.kv_caps[0], policies, deltas, cores, pool)
        tb_tot = tok_tot = 0
        t_tot = 0.0
        for _ in range(args.steps):
            tb, tok, dt, _ = oracle_timed(inputs, wl.B[0], wl.kv_caps[0], policies, deltas, cores, pool)
            tb_tot += tb
            tok_tot += tok
            t_tot += dt
    value = tb_tot / t_tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t_tot / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32",
        "data": "synthetic",
        "config": workload_config("cpu-oracle", wl, wl.n_instances, policies, deltas, "n/a (CPU)"),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"first {cores * per_core} of {wl.n_instances} instances x "
                                   f"{len(policies)} runs per step",
                         "cpu": cpu_model()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "token_advances_per_s": tok_tot / t_tot,
    }
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--kernel", choices=["step", "epoch"], default="step")
    ap.add_argument("--workload", type=int, choices=sorted(GRIDS), default=DEFAULT_WID)
    ap.add_argument("--instances", type=int, default=0, help="use only the first N instances (profiling)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-cores", type=int, default=0, help="host processes for the oracle (default: all cores)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-epoch", action="store_true", help="skip the event-driven kernel's extra measurement")
    args = ap.parse_args()
    if args.impl == "reference":
        return reference_arm(args)

    world, rank, local = dist_env()
    wid = args.workload
    wl = W.WORKLOADS[wid]
    policies, deltas, per_core = GRIDS[wid]
    n_inst = min(args.instances or wl.n_instances, wl.n_instances)
    B, kv = wl.B[0], wl.kv_caps[0]

    # the oracle pool starts before the first CUDA call (spawned workers)
    pool = None
    cores = args.oracle_cores or os.cpu_count() or 1
    if rank == 0 and not args.no_cpu_baseline:
        pool = mp.get_context("spawn").Pool(cores)

    import torch
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2608_02244_gb300 import sim

    a_h, p_h, o_h, c_h, e_h = host_inputs(wid, n_inst, replica=rank)
    a, p, o = (torch.from_numpy(x).cuda() for x in (a_h, p_h, o_h))
    cnt = torch.from_numpy(c_h).cuda() if c_h is not None else None
    slk = torch.from_numpy(e_h).cuda() if e_h is not None else None
    epoch = args.kernel == "epoch"
    S = sim.Simulator(n_inst, wl.n_per_instance, B, wl.c, wl.tau, wl.p0, epoch=epoch, timing=True)
    flush = torch.empty(64 * 2**20, dtype=torch.int32, device="cuda")   # 256 MiB > 129 MB L2
    stream = torch.cuda.current_stream()

    def sweep(simr):
        return simr.sweep_async(a, p, o, policies, deltas, kv, per_request=True, counts=cnt, slack=slk)

    # warm-up (also yields the deterministic per-step unit counts)
    for _ in range(max(args.warmup, 1)):
        sweep(S)
    st, summ = sim.isjl_sim_metrics(S.handle)
    if st != 0:
        raise RuntimeError(f"device status {st}: {sim.isjl_status_string(st)}")
    runs = [sim.summary_to_dict(summ[i]) for i in range(len(policies))]
    busy_per_step = sum(r["T_busy"] for r in runs)
    tok_per_step = sum(r["token_adv"] for r in runs)
    launches_per_step = sim.isjl_sim_last_launches(S.handle)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        uuid = None
    def timed_steps(simr):
        """K timed sweeps (L2 flushed before each, outside the events)."""
        sim_ms = []
        ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        t0 = time.perf_counter()
        for k in range(args.steps):
            flush.zero_()
            ev0[k].record(stream)
            sweep(simr)
            ev1[k].record(stream)
            sim_ms.append(sim.isjl_sim_kernel_times(simr.handle)[2])   # waits for this step's events
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        wall_s = time.perf_counter() - t0
        return [ev0[k].elapsed_time(ev1[k]) for k in range(args.steps)], sim_ms, wall_s

    sampler = ClockSampler(uuid)
    time.sleep(0.4)
    step_ms, sim_ms, wall = timed_steps(S)
    clocks = sampler.stop()
    t_ms = sum(step_ms)

    # the other kernel variant on the same inputs (same results), for comparison
    other = None
    if not args.no_epoch:
        S2 = sim.Simulator(n_inst, wl.n_per_instance, B, wl.c, wl.tau, wl.p0, epoch=not epoch, timing=True)
        for _ in range(max(args.warmup, 1)):
            sweep(S2)
        st2, summ2 = sim.isjl_sim_metrics(S2.handle)
        busy2 = sum(summ2[i].T_busy for i in range(len(policies)))
        if st2 != 0 or busy2 != busy_per_step:
            raise RuntimeError("kernel variants disagree")
        step2, sim2, _ = timed_steps(S2)
        other = {"kernel": "step" if epoch else "epoch",
                 "value": busy_per_step * args.steps / (sum(step2) / 1e3),
                 "ms_per_step": sum(step2) / args.steps, "sim_ms_per_launch": sum(sim2) / len(sim2)}
        S2.close()

    # e2e through the host-memory entry point: H2D of the inputs (and counts /
    # slack where the workload has them), sweep, D2H of the records
    e2e = None
    if not args.no_e2e:
        pa, pp, po = (torch.from_numpy(x).pin_memory() for x in (a_h, p_h, o_h))
        pc = torch.from_numpy(c_h).pin_memory() if c_h is not None else None
        pe = torch.from_numpy(e_h).pin_memory() if e_h is not None else None
        hrec = torch.empty(len(policies) * n_inst * sim.RECORD_DTYPE.itemsize, dtype=torch.uint8).pin_memory()

        def host_sweep():
            return sim.isjl_sim_run_sweep_host(S.handle, policies, deltas, kv, pa, pp, po, hrec, h_count=pc,
                                               h_slack=pe)
        host_sweep()   # warm
        torch.cuda.synchronize()
        e2e_ms = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            rc = host_sweep()
            e2e_ms.append(1e3 * (time.perf_counter() - t0))
            if rc != 0:
                raise RuntimeError(f"host sweep status {rc}")
        h2d = 3 * a_h.nbytes + (c_h.nbytes if c_h is not None else 0) + (e_h.nbytes if e_h is not None else 0)
        e2e = {"ms": sum(e2e_ms) / len(e2e_ms), "h2d": h2d, "d2h": hrec.numel()}

    # max over ranks, sum of units
    units = float(busy_per_step * args.steps)
    t_ms_all, units_all, e2e_ms_all = combine_ranks(t_ms, units, e2e["ms"] if e2e else 0.0, dist, "cuda")

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        S.close()
        return 0

    value = units_all / (t_ms_all / 1e3)
    sm_mhz = clocks.get("sm_mhz") or float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
                                            .get("clocks_under_load", {}).get("sm_mhz_median", 1417.0))
    sms = torch.cuda.get_device_properties(local).multi_processor_count
    nominal_tops = sms * ALU_LANES_PER_SM * sm_mhz * 1e6 / 1e12
    probe_sampler = ClockSampler(uuid)
    time.sleep(0.3)
    peaks = probe_peaks(sim, stream)
    probe_clocks = probe_sampler.stop()
    peak_tops = peaks["add"]
    # the event-driven kernel's own algorithmic work, counted from the outputs
    # of one sweep (starts and completions per request, distinct event steps)
    res = S.sweep(a, p, o, policies, deltas, kv, per_request=True, counts=cnt, slack=slk)
    st_h, co_h = res["start"], res["completion"]
    n_events = int((st_h >= 0).sum() + (co_h >= 0).sum())
    n_epochs = epoch_count(st_h, co_h)
    del res, st_h, co_h
    ops_step = OPS_PER_TOKEN_ADVANCE * tok_per_step + OPS_PER_BATCH_STEP * busy_per_step
    ops_epoch = OPS_PER_REQUEST_EVENT * n_events + OPS_PER_EPOCH * n_epochs

    def roof(kernel_name, ops, ms_per_launch, traffic):
        achieved = ops / (ms_per_launch / 1e3) / 1e12
        return {"bound": "alu", "achieved": achieved, "peak": peak_tops, "unit": "Tops/s",
                "frac": achieved / peak_tops, "traffic": traffic, "kernel": kernel_name,
                "ops_per_launch": ops, "sim_ms_per_launch": ms_per_launch,
                "peak_measured": peaks["add"], "alu_pipe_peak_measured": peaks["minmax"],
                "frac_of_alu_pipe": achieved / peaks["minmax"], "peak_nominal": nominal_tops,
                "peak_basis": (f"measured: isjl_probe_int_rate, int32 add chains ({peaks['add']:.2f} Tops/s) and "
                               f"min/max chains ({peaks['minmax']:.2f} Tops/s), best of {PROBE_LAUNCHES} "
                               f"full-occupancy launches at {probe_clocks.get('sm_mhz')} MHz; nominal "
                               f"{sms} SMs x {ALU_LANES_PER_SM} lanes x {sm_mhz:.0f} MHz = {nominal_tops:.2f}")}

    full = wid == DEFAULT_WID and n_inst == wl.n_instances
    sim_avg_ms = sum(sim_ms) / len(sim_ms)
    if epoch:
        roofline = roof("sim_kernel (epoch)", ops_epoch, sim_avg_ms, None)
    else:
        roofline = roof("sim_kernel (step)", ops_step, sim_avg_ms, SIM_DRAM_BYTES_PER_LAUNCH if full else None)
        if full:
            roofline["ncu_issue_active"] = SIM_NCU_ISSUE_ACTIVE
            roofline["ncu_alu_pipe"] = SIM_NCU_ALU_PIPE
    if other is not None:
        o_ops = ops_epoch if other["kernel"] == "epoch" else ops_step
        o_roof = roof(f"sim_kernel ({other['kernel']})", o_ops, other["sim_ms_per_launch"], None)
        other["roofline"] = {k: o_roof[k] for k in ("achieved", "frac", "frac_of_alu_pipe", "ops_per_launch")}
        other["epochs_per_launch"] = n_epochs
        other["request_events_per_launch"] = n_events

    cpu = None
    if pool is not None:
        sample_n = min(n_inst, cores * per_core)
        tb, tok, dt, used = oracle_timed(host_inputs(wid, sample_n, replica=rank), B, kv, policies, deltas,
                                         cores, pool)
        pool.close()
        cpu = {"value": tb / dt, "unit": UNIT, "cores": used, "kind": "oracle",
               "sample": f"first {sample_n} of {n_inst} instances x {len(policies)} runs ({dt:.1f} s wall)",
               "cpu": cpu_model()}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_ms_all / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int32", "data": "synthetic",
        "config": workload_config(args.kernel, wl, n_inst, policies, deltas,
                                  "flushed between steps (256 MiB write, outside the events)"),
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": ({"value": units_all / (e2e_ms_all / 1e3) / args.steps, "unit": UNIT,
                 "h2d_bytes_per_step": e2e["h2d"], "d2h_bytes_per_step": e2e["d2h"],
                 "outputs": "records only: the host entry point returns the per-(run, instance) records; "
                            "per-request start / completion steps are not copied back"} if e2e else None),
        "gpu_launches": launches_per_step * args.steps,
        "clocks": {"sm_mhz": clocks.get("sm_mhz"), "sm_max_mhz": clocks.get("sm_max_mhz"),
                   "reasons": clocks.get("reasons"), "probe_sm_mhz": probe_clocks.get("sm_mhz"),
                   "probe_reasons": probe_clocks.get("reasons")},
        "instances_per_s": world * n_inst * len(policies) * args.steps / (t_ms_all / 1e3),
        "token_advances_per_s": tok_per_step * world * args.steps / (t_ms_all / 1e3),
        "kernel_ms": {"sim": sim_avg_ms},
        "other_kernel": other,
        "wall_s": wall,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    S.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
