"""The seeded generator: determinism, per-instance addressability and ranges."""
import numpy as np
import pytest

from paper_2608_02244_gb300 import workloads as W


@pytest.mark.parametrize("wid", [1, 2, 3, 4])
def test_deterministic_and_addressable(wid):
    wl = W.WORKLOADS[wid]
    ids = [0, min(3, wl.n_instances - 1)]
    a1 = W.generate(wid, ids)
    a2 = W.generate(wid, ids)
    for x, y in zip(a1, a2):
        np.testing.assert_array_equal(x, y)
    single = W.generate(wid, [ids[-1]])
    for x, y in zip(a1, single):
        np.testing.assert_array_equal(x[-1], y[0])
    for x in a1:
        assert x.dtype == np.int32 and x.shape == (len(ids), wl.n_per_instance)


def test_ranges():
    a, p, o = W.generate(1)
    assert (a == 0).all() and p.min() >= 1 and p.max() <= 32
    assert set(np.unique(o)) <= set(range(1, 17)) | set(range(64, 257))
    a, p, o = W.generate(2)
    assert a.shape == (4096, 6) and p.min() >= 1 and p.max() <= 4 and o.min() >= 1 and o.max() <= 8
    a, p, o = W.generate(3, 8)
    assert (np.diff(a, axis=1) >= 0).all() and a.min() >= 0
    assert p.min() >= 16 and p.max() <= 4096 and o.min() >= 1 and o.max() <= 2048
    a, p, o = W.generate(4, 8)
    assert (a == 0).all() and p.min() >= 16 and p.max() <= 1024 and o.min() >= 8 and o.max() <= 8192
    a, p, o = W.generate(5, [0])
    assert (np.diff(a, axis=1) >= 0).all() and p.min() >= 16 and p.max() <= 32768 and o.max() <= 16384
    # mean gap 0.05: 1e5 requests arrive within a few thousand steps
    assert 4000 < a[0, -1] < 6000

