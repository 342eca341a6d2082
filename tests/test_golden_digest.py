"""The stored oracle digests of the large-instance workload stay in step with
the oracle and the workload generator (CPU only).

tests/golden/large_instance_digest.txt holds, per instance, a digest of the
generated inputs and of the oracle's integer record fields and per-request
steps (written by tests/golden/make_large_digest.py).  Here: the file covers
every instance once, and instance 0's digests are recomputed from scratch.
"""
import importlib.util
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _module():
    spec = importlib.util.spec_from_file_location("make_large_digest",
                                                  os.path.join(GOLDEN, "make_large_digest.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _stored():
    rows = {}
    with open(os.path.join(GOLDEN, "large_instance_digest.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            i, din, dres = line.split()
            assert int(i) not in rows
            rows[int(i)] = (din, dres)
    return rows


def test_digest_file_covers_every_instance():
    from paper_2608_02244_gb300 import workloads as W
    D = _module()
    rows = _stored()
    assert sorted(rows) == list(range(W.WORKLOADS[D.WID].n_instances))
    assert all(len(d) == 16 and len(r) == 16 for d, r in rows.values())


def test_first_instance_recomputed_with_the_oracle():
    from oracle import oracle as O
    from paper_2608_02244_gb300 import workloads as W
    D = _module()
    rows = _stored()
    wl = W.WORKLOADS[D.WID]
    a, p, o = W.generate(D.WID, instances=[0, wl.n_instances - 1])
    assert D.input_digest(a[1], p[1], o[1]) == rows[wl.n_instances - 1][0]
    assert D.input_digest(a[0], p[0], o[0]) == rows[0][0]
    res = [O.run(pol, wl.B[0], d, wl.kv_caps[0], a[:1], p[:1], o[:1], per_request=True) for pol, d in D.RUNS]
    got = D.result_digest([r[0][0] for r in res], [r[1][0] for r in res], [r[2][0] for r in res])
    assert got == rows[0][1]
    # the digest sees every field: one changed step gives another digest
    st = [r[1][0].copy() for r in res]
    st[2][int(np.argmax(st[2]))] += 1
    assert D.result_digest([r[0][0] for r in res], st, [r[2][0] for r in res]) != got
