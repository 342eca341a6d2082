"""GB300-native batched simulator of FCFS, LJF and ISJL scheduling.

Simulates the token-step serving model of "Efficiency and Cost Alignment in
Batched LLM Serving via Resource-Fair Scheduling" over many request instances
and fairness budgets on one GPU.  The work runs in hand-written sm_103a CUDA
kernels behind the C ABI of ``include/isjl_sim.h``; ``sim`` is the Python
binding and ``workloads`` draws seeded synthetic instances.
"""
from . import workloads  # noqa: F401

__all__ = ["workloads", "sim", "build"]
