"""CUDA path of the paper's literal per-message B-FASGD (mean-v decision,
server gradient cache) against the oracle."""

import numpy as np
import pytest

import oracle
from gpu_util import CudaRun, OracleRun, assert_bitwise, compare_states
from paper_1601_04033_gb300 import streams

pytestmark = pytest.mark.gpu

SEED = 0x3E55A6E


def _run_pair(P, n_push, c_push, lam=3, variant=oracle.FASGD):
    import torch
    w = streams.WORKLOADS["fasgd-1.29m"].replace(lam=lam, R=8)
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w, n_push, 1)
    g = CudaRun(w, variant, P, pool, th0, c_push=c_push, seed=SEED)
    o = OracleRun(w, variant, P, pool, th0, c_push=c_push, seed=SEED)
    flags = torch.full((n_push,), -1, dtype=torch.int32, device="cuda")
    for t in range(n_push):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.push_message(c, j, g.pool[s], sent_dev=flags[t:t + 1])
        g.srv.apply_pending(1)
        o.srv.push_message(c, j, pool[s])
        o.srv.apply_pending(1)
        if (t + 1) % 100 == 0:
            compare_states(g.state(), o.state(), variant, f"message T={t + 1}")
    got = flags.cpu().numpy()
    assert np.array_equal(got, np.array(o.srv.message_log, dtype=np.int32)), "decisions differ"
    return g, o, got


@pytest.mark.parametrize("P", [5, 8192, 70_001])
def test_message_pushes_against_oracle(P):
    # c chosen so that roughly half the pushes are transmitted once v settles
    _, _, flags = _run_pair(P, 200, 40.0)
    assert 0 < flags.sum() < flags.size


def test_message_c0_equals_dense_and_cinf_applies_zeros():
    import torch
    w = streams.WORKLOADS["fasgd-1.29m"].replace(lam=2, R=4)
    P = 10_007
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w, 30, 1)
    a = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=0.0, seed=SEED)
    b = CudaRun(w, oracle.FASGD, P, pool, th0)
    z = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=float("inf"), seed=SEED)
    zb = CudaRun(w, oracle.FASGD, P, np.zeros_like(pool), th0)
    for t in range(30):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        a.srv.push_message(c, j, a.pool[s])
        a.srv.apply_pending(1)
        b.push_batch(cl, js, sl)
        z.srv.push_message(c, j, z.pool[s])
        z.srv.apply_pending(1)
        zb.push_batch(cl, js, sl)
    for x, y in zip(a.state()[:4], b.state()[:4]):
        assert_bitwise(x, y, "c=0")
    for x, y in zip(z.state()[:4], zb.state()[:4]):
        assert_bitwise(x, y, "c=inf")
    # a message push under FASGD: the statistic's partials, then the pass that
    # decides, refreshes the cache slot and applies
    assert a.srv.launches == 30 * 2 and b.srv.launches == 30


def test_fetch_messages_against_oracle():
    import torch
    from paper_1601_04033_gb300 import fasgd
    P = 33_333
    rng = np.random.default_rng(12)
    theta = (rng.standard_normal(P) * 0.01).astype(np.float32)
    n = np.zeros(P, np.float32)
    b = np.zeros(P, np.float32)
    v = (10 ** rng.uniform(0, 2, P)).astype(np.float32)
    srv = fasgd.Server(P, 3, 0.001, fasgd.FASGD, seed=SEED)
    srv.set_state(*[torch.from_numpy(x).cuda() for x in (theta, n, b, v)], 5)
    o = oracle.OracleServer(P, 3, 0.001, oracle.FASGD, seed=SEED)
    o.theta[:], o.n[:], o.b[:], o.v[:] = theta, n, b, v
    vbar = oracle.mean_v(v)
    for c in (0.0, vbar, float("inf")):            # always, about half, never
        srv.set_fetch_threshold(c)
        o.set_fetch_threshold(c)
        for k in range(40):
            client = k % 3
            gcopy = torch.full((P,), 7.0, device="cuda")
            flag = torch.full((1,), -1, dtype=torch.int32, device="cuda")
            srv.fetch_message(client, gcopy, fetched_dev=flag)
            ocopy = np.full(P, 7.0, np.float32)
            ok = o.fetch_message(client, ocopy)
            assert int(flag.item()) == int(ok), (c, k)
            assert_bitwise(gcopy.cpu().numpy(), ocopy, f"fetched copy c={c} k={k}")
    assert list(srv.fetch_counts()) == o.fetch_count


@pytest.mark.parametrize("P", [5, 2048 * 3 + 129, 100_003, 300_000])
def test_statistic_kept_by_the_dense_pass_equals_a_fresh_sum(P):
    """After a message push the dense pass leaves the chunk sums of the new v;
    the statistic formed from them equals, bit for bit, the one formed afresh
    from v (after set_state, which discards the kept sums), and equals the
    oracle's mean of v.  Sizes cover the dense pass's tail (P mod 2048, 128, 4)."""
    import torch
    from paper_1601_04033_gb300 import fasgd
    w = streams.WORKLOADS["fasgd-1.29m"].replace(lam=3, R=4)
    pool = streams.gradient_pool(w, P)
    srv = fasgd.Server(P, 3, w.alpha, fasgd.FASGD, c_push=1.0, seed=SEED)
    srv.set_params(torch.from_numpy(streams.theta0(w, P)).cuda())
    _, dpool = fasgd.aligned_vectors(pool)
    state = [torch.empty(P, device="cuda") for _ in range(4)]
    for t in range(6):
        if t == 3:                      # a fused dense pass in between (it discards the sums)
            srv.push(0, srv.T, dpool[1])
            srv.push(1, srv.T, dpool[2])
            srv.apply_pending(2)
        srv.push_message(t % 3, srv.T, dpool[t % 4])
        srv.apply_pending(1)
        kept = srv.message_vbar()
        T = srv.get_state(*state)
        srv.set_state(*state, T)
        fresh = srv.message_vbar()
        assert np.float32(kept).view(np.uint32) == np.float32(fresh).view(np.uint32), (t, kept, fresh)
        assert fresh == oracle.mean_v(state[3].cpu().numpy()), (t, fresh)


@pytest.mark.slow
def test_full_size_25m_messages():
    """P = 25,000,000 (the benchmark's message workload, 4 clients): 10 message
    pushes and 10 message fetches, every decision equal to the oracle's, the
    statistic kept by the dense pass equal to a fresh sum at the end, and the
    state on sampled parameters."""
    import torch
    from paper_1601_04033_gb300 import fasgd
    w = streams.WORKLOADS["bfasgd-message-25m"].replace(lam=4, R=4)
    P = w.P
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=2.0, seed=SEED)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, c_push=2.0, seed=SEED)
    g.srv.set_fetch_threshold(4.0)
    o.srv.set_fetch_threshold(4.0)
    flag = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    sent = torch.full((10,), -1, dtype=torch.int32, device="cuda")
    ps = streams.push_stream(w, 10, 1)
    fetched = []
    for t in range(10):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.push_message(c, j, g.pool[s], sent_dev=sent[t:t + 1])
        g.srv.apply_pending(1)
        o.srv.push_message(c, j, pool[s])
        o.srv.apply_pending(1)
        copy = torch.zeros(P, device="cuda")
        g.srv.fetch_message(c, copy, fetched_dev=flag)
        ok = o.srv.fetch_message(c, np.zeros(P, np.float32))
        assert int(flag.item()) == int(ok), f"fetch {t}"
        fetched.append(ok)
    assert g.srv.fetch_counts().tolist() == o.srv.fetch_count
    kept = g.srv.message_vbar()
    gs = g.state()
    assert np.array_equal(sent.cpu().numpy(), np.array(o.srv.message_log, dtype=np.int32))
    assert 0 < sum(o.srv.message_log) < 10 or 0 < sum(fetched) < 10
    state = [torch.from_numpy(x).cuda() for x in gs[:4]]
    g.srv.set_state(*state, gs[4])
    fresh = g.srv.message_vbar()
    assert np.float32(kept).view(np.uint32) == np.float32(fresh).view(np.uint32)
    assert fresh == oracle.mean_v(gs[3])
    idx = streams.sample_indices(P, 50_000)
    os_ = o.state()
    compare_states([x[idx] for x in gs[:4]] + [gs[4]], [x[idx] for x in os_[:4]] + [os_[4]],
                   oracle.FASGD, "25M messages")


@pytest.mark.slow
def test_message_vbar_bits_at_25m():
    """The per-message statistic (Sec. 2.3: the mean of v over every parameter)
    at P = 25,000,000, bit for bit against the oracle's exact mean, on v
    spread over six decades, with zeros mixed in, and on v of two adjacent
    floats (a mean that sits between them)."""
    import torch
    from paper_1601_04033_gb300 import fasgd
    P = 25_000_000
    rng = np.random.default_rng(2525)
    srv = fasgd.Server(P, 2, 0.001, fasgd.FASGD, seed=SEED)
    zeros = torch.zeros(P, device="cuda")
    lo = np.float32(0.3)
    cases = [
        (10 ** rng.uniform(-3, 3, P)).astype(np.float32),
        np.where(rng.random(P) < 0.3, 0.0, 10 ** rng.uniform(-2, 2, P)).astype(np.float32),
        np.where(rng.random(P) < 0.5, lo, np.nextafter(lo, np.float32(1))).astype(np.float32),
    ]
    for k, v in enumerate(cases):
        srv.set_state(zeros, zeros, zeros, torch.from_numpy(v).cuda(), 0)
        got = srv.message_vbar()
        want = oracle.mean_v(v)
        assert np.float32(got).view(np.uint32) == np.float32(want).view(np.uint32), (k, got, want)
    srv.close()
