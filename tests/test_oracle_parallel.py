"""The process-pool runner of the oracle (test infrastructure for the
whole-workload parity tests and the benchmark's CPU legs)."""
import numpy as np

from paper_2608_02244_gb300 import workloads as W


def test_parallel_oracle_equals_serial():
    """oracle.parallel splits instances over a spawned pool and concatenates
    the blocks back in order: the same records and per-request steps as one
    serial call, with and without ragged counts and slack."""
    from oracle import oracle as O, parallel
    a, p, o, cnt, e = W.generate(6, 9, with_counts=True, with_slack=True)
    e = (e + 3).astype(np.int32)
    pool = parallel.make_pool(2)
    try:
        for pol, d in (("isjl", 150), ("fcfs", 0)):
            r0, s0, c0 = O.run(pol, 50, d, 2**31 - 1, a, p, o, counts=cnt, slack=e)
            r1, s1, c1 = parallel.run(pool, pol, 50, d, 2**31 - 1, a, p, o, per_request=True, counts=cnt, slack=e,
                                      block=2)
            assert r0.tobytes() == r1.tobytes()
            np.testing.assert_array_equal(s0, s1)
            np.testing.assert_array_equal(c0, c1)
    finally:
        pool.close()
        pool.join()
