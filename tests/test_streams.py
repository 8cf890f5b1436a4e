"""The seeded workload generator (no GPU)."""

import numpy as np

from paper_1601_04033_gb300 import streams


def test_deterministic_and_distinct_slots():
    w = streams.WORKLOADS["fasgd-25m-k8"].replace(P=1000)
    a = streams.push_stream(w, 400)
    b = streams.push_stream(w, 400)
    assert np.array_equal(a.j, b.j) and np.array_equal(a.slot, b.slot)
    for k in range(400 // w.K):
        _, _, sl = a.batch(k)
        assert len(set(sl.tolist())) == w.K
    assert np.array_equal(streams.gradient_pool(w, 1000, 3), streams.gradient_pool(w, 1000, 3))


def test_timestamps_legal():
    for name, w in streams.WORKLOADS.items():
        n = 2000
        ps = streams.push_stream(w, n)
        Tb = (np.arange(n) // w.K) * w.K
        assert np.all(ps.j >= 0) and np.all(ps.j <= Tb), name
        assert np.all(ps.client >= 0) and np.all(ps.client < w.lam)


def test_delay_laws():
    w = streams.WORKLOADS
    d = streams.delays(w["fasgd-7850"], 20000)
    assert d.min() == 0 and d.max() == 3
    assert abs(streams.delays(w["fasgd-1.29m"], 20000).mean() - 4) < 0.1
    assert abs(streams.delays(w["bfasgd-25m"], 20000).mean() - 8) < 0.15
    g = streams.delays(w["fasgd-25m-k8"], 20000)
    assert g.min() == 0 and g.max() <= 512 and abs(g.mean() - 19) < 1.0   # (1-p)/p = 19
    p = streams.delays(w["fasgd-268m-k16"], 20000)
    assert p.min() == 0 and p.max() <= 4096


def test_gradient_model_ranges():
    w = streams.WORKLOADS["fasgd-7850"]
    m, s = streams.grad_model(w)
    assert m.dtype == np.float32 and s.dtype == np.float32
    assert abs(m.std() - 1e-3) < 1e-4
    assert s.min() >= 1e-4 * 0.999 and s.max() <= 1e-1 * 1.001
    th = streams.theta0(w)
    assert abs(th.std() - 0.01) < 1e-3
    v = streams.client_v_snapshot(w, 2)
    assert v.min() >= 1.0 and v.max() <= 100.0
