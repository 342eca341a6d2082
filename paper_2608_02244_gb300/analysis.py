"""Post-processing of simulation records (host side, numpy).

These helpers consume the per-(run, instance) records the CUDA path returns;
they are not steps of the simulation.

  cost_table       Table 1 quantities of Section 5.2 per policy: profit, cost
                   and its terms tau*Q, c*T, tau*E (Theorem "Profit
                   decomposition"), throughput, gain vs LJF, average extent
  break_even_c     Table 2: c*_alpha = tau E_ISJL / (T_LJF - T_ISJL), the fixed
                   step cost above which ISJL out-earns LJF (Prop. "Pairwise
                   profit comparison"); None when ISJL is not faster
  alpha_cost       alpha_cost(delta) = delta * Q / O (Section 5.1): every
                   alpha-fair schedule then has tau E <= delta tau Q
  calibrate_alpha  alpha* = argmin over a grid of c T + tau E, optionally
                   subject to a throughput floor and a latency-quantile cap
                   (Section 5.1's calibration procedure); ties to the smaller alpha
"""
from __future__ import annotations

import numpy as np

TABLE1_FIELDS = ("profit", "cost", "tau_Q", "c_T", "tau_E", "throughput", "avg_extent")


def avg_extent(records):
    """Mean over nonempty steps of max r - min r, per record."""
    tb = np.asarray(records["T_busy"], dtype=np.float64)
    return np.where(tb > 0, np.asarray(records["sum_extent"], dtype=np.float64) / np.maximum(tb, 1), 0.0)


def cost_table(records_by_key, ljf_key=None):
    """Means over instances of the Table 1 columns, per key (e.g. (policy, alpha)).

    ``records_by_key`` maps a key to a structured record array (one record per
    instance).  With ``ljf_key`` the result also carries the throughput gain
    relative to that key's mean throughput, in percent.
    """
    out = {}
    for key, rec in records_by_key.items():
        row = {f: float(np.mean(rec[f])) for f in TABLE1_FIELDS if f != "avg_extent"}
        row["avg_extent"] = float(np.mean(avg_extent(rec)))
        row["T_make"] = float(np.mean(rec["T_make"]))
        out[key] = row
    if ljf_key is not None:
        base = out[ljf_key]["throughput"]
        for row in out.values():
            row["gain_vs_ljf_pct"] = 100.0 * (row["throughput"] / base - 1.0)
    return out


def break_even_c(tau_E_isjl, T_ljf, T_isjl):
    """c* = tau E_ISJL / (T_LJF - T_ISJL); None unless ISJL's makespan is shorter."""
    gap = float(T_ljf) - float(T_isjl)
    if gap <= 0:
        return None
    return float(tau_E_isjl) / gap


def alpha_cost(delta_frac, Q, O):
    """Largest budget whose externality bound E <= alpha O stays within delta Q."""
    return float(delta_frac) * float(Q) / float(O)


def calibrate_alpha(alphas, c_T, tau_E, throughput=None, throughput_sla=None, latency_q=None, latency_sla=None):
    """alpha* = argmin_alpha c T + tau E over the grid, among alphas meeting the
    optional throughput floor and latency-quantile cap.  Returns None if no
    alpha qualifies.  Ties go to the smaller alpha (tighter cost alignment)."""
    alphas = np.asarray(alphas)
    obj = np.asarray(c_T, dtype=np.float64) + np.asarray(tau_E, dtype=np.float64)
    ok = np.ones(alphas.shape, bool)
    if throughput_sla is not None:
        ok &= np.asarray(throughput, dtype=np.float64) >= throughput_sla
    if latency_sla is not None:
        ok &= np.asarray(latency_q, dtype=np.float64) <= latency_sla
    if not ok.any():
        return None
    order = np.lexsort((alphas, obj))          # by objective, then by alpha
    for i in order:
        if ok[i]:
            return alphas[i].item()
    return None
