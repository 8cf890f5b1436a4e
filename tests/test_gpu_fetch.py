"""CUDA B-FASGD fetch path (per-parameter fetch decision + compaction of theta,
client-side scatter) against the oracle."""

import numpy as np
import pytest

import oracle
from gpu_util import CudaRun, OracleRun, assert_bitwise, assert_close, compare_states
from paper_1601_04033_gb300 import streams
from paper_1601_04033_gb300.calibrate import calibrate_c

pytestmark = pytest.mark.gpu

SEED = 0x0FE7C4
EPS_B = 1e-8


def _f():
    from paper_1601_04033_gb300 import fasgd
    return fasgd


def _lists(P):
    import torch
    return (torch.full((P,), -1, dtype=torch.int32, device="cuda"),
            torch.full((P,), float("nan"), device="cuda"),
            torch.full((1,), -1, dtype=torch.int64, device="cuda"))


def _state(P, seed):
    rng = np.random.default_rng(seed)
    theta = (rng.standard_normal(P) * 0.01).astype(np.float32)
    n = (10 ** rng.uniform(-6, -2, P)).astype(np.float32)
    b = (rng.standard_normal(P) * 1e-3).astype(np.float32)
    v = (10 ** rng.uniform(0, 2, P)).astype(np.float32)
    return theta, n, b, v


@pytest.mark.parametrize("P", [1, 5, 8191, 8193, 100_003])
def test_fetch_compact_bit_exact(P):
    import torch
    f = _f()
    theta, n, b, v = _state(P, P)
    srv = f.Server(P, 4, 0.001, f.FASGD, eps_b=EPS_B, seed=SEED)
    srv.set_state(*[torch.from_numpy(x).cuda() for x in (theta, n, b, v)], 17)
    for c in (0.0, calibrate_c(v, 0.1), float("inf")):
        srv.set_fetch_threshold(c)
        for k in range(2):
            idx, val, cnt = _lists(P)
            srv.fetch_compact(3, idx, val, cnt)                  # live v
            m = int(cnt.item())
            oi, ov = oracle.fetch_select(theta, v, np.float32(c), EPS_B, SEED, 3,
                                         int(srv.fetch_counts()[3]) - 1)
            assert m == oi.size
            assert_bitwise(idx[:m].cpu().numpy(), oi, f"fetch idx P={P} c={c}")
            assert_bitwise(val[:m].cpu().numpy(), ov, f"fetch val P={P} c={c}")
    assert list(srv.push_counts()) == [0, 0, 0, 0]
    srv.close()


def test_fetch_and_push_streams_differ():
    import torch
    f = _f()
    P = 50_000
    theta, n, b, v = _state(P, 1)
    srv = f.Server(P, 2, 0.001, f.FASGD, c_push=5.0, eps_b=EPS_B, seed=SEED)
    srv.set_state(*[torch.from_numpy(x).cuda() for x in (theta, n, b, v)], 0)
    srv.set_fetch_threshold(5.0)
    th = torch.from_numpy(theta).cuda()
    a = _lists(P)
    b_ = _lists(P)
    srv.select_compact(1, th, *a)          # push decision over the same values
    srv.fetch_compact(1, *b_)
    ma, mb = int(a[2].item()), int(b_[2].item())
    ia, ib = a[0][:ma].cpu().numpy(), b_[0][:mb].cpu().numpy()
    assert not np.array_equal(ia, ib)
    assert list(srv.push_counts()) == [0, 1] and list(srv.fetch_counts()) == [0, 1]


def test_fetch_apply_matches_oracle_and_flags_bad_indices():
    import torch
    f = _f()
    P = 30_011
    theta, n, b, v = _state(P, 3)
    srv = f.Server(P, 2, 0.001, f.FASGD, eps_b=EPS_B, seed=SEED)
    srv.set_state(*[torch.from_numpy(x).cuda() for x in (theta, n, b, v)], 0)
    srv.set_fetch_threshold(calibrate_c(v, 0.3))
    idx, val, cnt = _lists(P)
    srv.fetch_compact(0, idx, val, cnt)
    stale = np.random.default_rng(4).standard_normal(P).astype(np.float32)
    client = torch.from_numpy(stale).cuda()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    f.fetch_apply(client, idx, val, n_dev=cnt, n_max=P, err_dev=err)
    m = int(cnt.item())
    ref = stale.copy()
    oracle.fetch_apply(ref, idx[:m].cpu().numpy(), val[:m].cpu().numpy())
    torch.cuda.synchronize()
    assert_bitwise(client.cpu().numpy(), ref, "client theta after fetch")
    assert int(err.item()) == 0
    bad = torch.tensor([0, P, -1, 5], dtype=torch.int32, device="cuda")
    f.fetch_apply(client, bad, torch.ones(4, device="cuda"), err_dev=err)
    torch.cuda.synchronize()
    assert int(err.item()) & 2
    got = client.cpu().numpy()
    assert got[0] == 1.0 and got[5] == 1.0
    # host-side argument checks
    with pytest.raises(f.FasgdError):
        f.fetch_apply(client, bad, torch.ones(4, device="cuda"), n_max=P + 1)


def test_bfasgd_round_trip_against_oracle():
    """Clients push through select/compact + sparse apply and refresh their
    stale copies through fetch/compact + scatter; both directions decide on
    drawn v snapshots so that CUDA and oracle take identical decisions."""
    import torch
    f = _f()
    w = streams.WORKLOADS["bfasgd-25m"].replace(lam=4, R=8)
    P = 60_007
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    vs = [streams.client_v_snapshot(w, c, P) for c in range(w.lam)]
    c_push = calibrate_c(vs[0], 0.2)
    c_fetch = calibrate_c(vs[0], 0.1)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    g.srv.set_fetch_threshold(c_fetch)
    o.srv.set_fetch_threshold(c_fetch)
    vs_t = [torch.from_numpy(x).cuda() for x in vs]
    gclients = [torch.from_numpy(th0.copy()).cuda() for _ in range(w.lam)]
    oclients = [th0.copy() for _ in range(w.lam)]
    ps = streams.push_stream(w, 120, 1)
    for t in range(120):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        idx, val, cnt = _lists(P)
        g.srv.select_compact(c, g.pool[s], idx, val, cnt, v=vs_t[c])
        g.srv.push_sparse(c, j, idx, val, n_dev=cnt, n_max=P)
        g.srv.apply_pending(1)
        oi, ov = o.srv.select_compact(c, pool[s], vs[c])
        o.srv.push_sparse(c, j, oi, ov)
        o.srv.apply_pending(1)
        fi, fv, fc = _lists(P)
        g.srv.fetch_compact(c, fi, fv, fc, v=vs_t[c])
        f.fetch_apply(gclients[c], fi, fv, n_dev=fc, n_max=P)
        oi2, ov2 = o.srv.fetch_compact(c, vs[c])
        oracle.fetch_apply(oclients[c], oi2, ov2)
        m = int(fc.item())
        assert_bitwise(fi[:m].cpu().numpy(), oi2, f"fetch idx t={t}")
        if (t + 1) % 40 == 0:
            compare_states(g.state(), o.state(), oracle.FASGD, f"round trip T={t + 1}")
            for k in range(w.lam):
                assert_close(gclients[k].cpu().numpy(), oclients[k], f"client {k} theta")
    g.srv.sync()
