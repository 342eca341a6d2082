"""The allocation-free sweep against the regular one.

isjl_sim_run_sweep_noalloc serves callers that cannot allocate device memory
where they need a simulation (allocator-owned pools, fixed budgets, sections
that must not synchronize): its workspace is a fixed device array shared by
every call.  Two calls in a row must each match the regular entry point, so
a stale workspace from the previous call cannot leak into the next.  This
file is collected last on purpose.
"""
import numpy as np
import pytest

from conftest import cuda_available

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not cuda_available(), reason="needs a CUDA GPU")]

INF = 2**31 - 1
F64 = ("c_T", "tau_Q", "tau_E", "cost", "revenue", "profit", "throughput", "ael")


def _check_equal(g, r):
    for f in r.dtype.names:
        if f in F64:
            np.testing.assert_allclose(g[f], r[f], rtol=1e-12, atol=0, err_msg=f)
        else:
            np.testing.assert_array_equal(g[f], r[f], err_msg=f)


@pytest.mark.parametrize("epoch", [False, True])
def test_noalloc_matches_regular_sweep_twice(epoch):
    import torch
    from paper_2608_02244_gb300 import sim, workloads as W
    cases = [
        (3, 24, 256, 200_000, ["fcfs", "ljf", "isjl", "isjl", "isjl"], [0, 0, 16, 256, INF]),
        (1, None, 32, 2048, ["fcfs", "ljf", "isjl"], [32, 32, 32]),
    ]
    flags = sim.FLAG_EPOCH_KERNEL if epoch else sim.FLAG_STEP_KERNEL
    for wid, count, B, kv, pols, ds in cases:
        a_h, p_h, o_h = W.generate(wid, count)
        n_inst, n = a_h.shape
        ref = sim.Simulator(n_inst, n, B, epoch=epoch)
        try:
            want = ref.sweep(a_h, p_h, o_h, pols, ds, kv, per_request=True)
        finally:
            ref.close()
        a, p, o = (torch.from_numpy(x).cuda() for x in (a_h, p_h, o_h))
        for _ in range(2):   # the second call runs on the first call's leftover workspace
            rec = torch.zeros(len(pols) * n_inst * sim.RECORD_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
            st = torch.full((len(pols) * n_inst * n,), -7, dtype=torch.int32, device="cuda")
            co = torch.full_like(st, -7)
            rc = sim.isjl_sim_run_sweep_noalloc(n_inst, n, B, pols, ds, kv, a, p, o, rec, st, co, flags=flags)
            assert rc == sim.ISJL_OK, sim.isjl_status_string(rc)
            torch.cuda.synchronize()
            got = sim.records_to_numpy(rec, len(pols), n_inst)
            for i in range(len(pols)):
                _check_equal(got[i], want["records"][i])
            np.testing.assert_array_equal(st.cpu().numpy().reshape(len(pols), n_inst, n), want["start"])
            np.testing.assert_array_equal(co.cpu().numpy().reshape(len(pols), n_inst, n), want["completion"])


@pytest.mark.parametrize("epoch", [False, True])
def test_noalloc_fewer_blocks_and_slack(epoch):
    """Large instances (n = 100,000): the fixed array holds the plan scratch of
    fewer simulation blocks than are resident, so the call runs on fewer
    warps; and a robust workload, whose true lengths take 4 more bytes per
    request.  Both must match the regular sweep, records and per-request steps."""
    import torch
    from paper_2608_02244_gb300 import sim, workloads as W
    flags = sim.FLAG_EPOCH_KERNEL if epoch else sim.FLAG_STEP_KERNEL
    cases = [(5, 3, 512, 1_000_000, ["fcfs", "isjl"], [0, 256], False),
             (8, 12, 256, 200_000, ["fcfs", "ljf", "isjl", "isjl"], [0, 0, 64, INF], True)]
    for wid, count, B, kv, pols, ds, robust in cases:
        a_h, p_h, o_h, _, e_h = W.generate(wid, count, with_counts=True, with_slack=True)
        e_h = e_h if robust else None
        n_inst, n = a_h.shape
        if wid == 5:   # the plan scratch of the resident blocks does not fit: fewer blocks run
            free = (64 << 20) - n_inst * n * 20 - 4096
            assert free // (4 * n) < 4 * 152
        ref = sim.Simulator(n_inst, n, B, epoch=epoch)
        try:
            want = ref.sweep(a_h, p_h, o_h, pols, ds, kv, per_request=True, slack=e_h)
        finally:
            ref.close()
        a, p, o = (torch.from_numpy(x).cuda() for x in (a_h, p_h, o_h))
        e = torch.from_numpy(e_h).cuda() if e_h is not None else None
        rec = torch.zeros(len(pols) * n_inst * sim.RECORD_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
        st = torch.full((len(pols) * n_inst * n,), -7, dtype=torch.int32, device="cuda")
        co = torch.full_like(st, -7)
        rc = sim.isjl_sim_run_sweep_noalloc(n_inst, n, B, pols, ds, kv, a, p, o, rec, st, co, flags=flags, slack=e)
        assert rc == sim.ISJL_OK, sim.isjl_status_string(rc)
        torch.cuda.synchronize()
        got = sim.records_to_numpy(rec, len(pols), n_inst)
        for i in range(len(pols)):
            _check_equal(got[i], want["records"][i])
        np.testing.assert_array_equal(st.cpu().numpy().reshape(len(pols), n_inst, n), want["start"])
        np.testing.assert_array_equal(co.cpu().numpy().reshape(len(pols), n_inst, n), want["completion"])


def test_noalloc_rejects_oversize_problem():
    import torch
    from paper_2608_02244_gb300 import sim
    x = torch.zeros(8, dtype=torch.int32, device="cuda")
    rec = torch.zeros(sim.RECORD_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    # 4 arrays x 4 bytes x 2**22 requests alone exceed the fixed 64 MiB workspace
    rc = sim.isjl_sim_run_sweep_noalloc(1 << 14, 1 << 8, 32, ["fcfs"], [0], 100, x, x, x, rec)
    assert rc == sim.ISJL_ERR_INVALID_ARG
