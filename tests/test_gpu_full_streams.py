"""Parity over each workload's whole push stream (Sec. 2.1 protocol, Eq. 1-2
and Eq. 4-8 applied push after push).  theta accumulates the rounding of
every step, so drift can only show over the full length of a stream, not a
prefix: the CUDA path (default fast arithmetic) is held to the oracle at
every T that is a multiple of lcm(100, K), to the end of the stream.

At P = 25M and 2^28 the oracle runs on sampled parameters alone: the update
is elementwise, so that sub-problem is exact.  The B-FASGD stream compares
every push's list bit for bit and the whole state every 100 pushes; the
per-message and per-tensor rules (Sec. 2.3 and Sec. 5) compare every
decision and the state every 100 pushes over the same 10,000-push stream."""

import math

import numpy as np
import pytest

import oracle
from gpu_util import CudaRun, OracleRun, assert_bitwise, compare_states, run_parity
from paper_1601_04033_gb300 import streams
from paper_1601_04033_gb300.calibrate import calibrate_c

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

W = streams.WORKLOADS


@pytest.mark.parametrize("variant", [oracle.ASGD, oracle.SASGD, oracle.FASGD])
def test_workload_1_29m_full_stream(variant):
    """P = 1,290,510, lambda = 32, Poisson(4) staleness, K = 1: all 10,000
    pushes, every parameter compared every 100 pushes."""
    w = W["fasgd-1.29m"]
    run_parity(w, variant, w.P, w.pushes, 1)


def _sampled_stream(w, P, n_pushes, K, R=None):
    """GPU at full size and the oracle on sampled parameters, in lockstep;
    the sampled state compared at every T multiple of lcm(100, K)."""
    import torch
    R = R or w.R
    wr = w.replace(R=R)
    pool = streams.gradient_pool(wr, P)
    th0 = streams.theta0(wr, P)
    ps = streams.push_stream(wr, n_pushes, K)
    idx = streams.sample_indices(P, 20_000)
    g = CudaRun(wr, oracle.FASGD, P, pool, th0)
    o = OracleRun(wr, oracle.FASGD, idx.size, np.ascontiguousarray(pool[:, idx]), th0[idx])
    del pool
    idx_t = torch.from_numpy(idx).cuda()
    full = [torch.empty(P, device="cuda") for _ in range(4)]
    every = 100 * K // math.gcd(100, K)
    checks = 0
    for b in range(n_pushes // K):
        batch = ps.batch(b)
        g.push_batch(*batch)
        o.push_batch(*batch)
        if ((b + 1) * K) % every == 0:
            T = g.srv.get_state(*full)
            gs = [x[idx_t].cpu().numpy() for x in full] + [T]
            compare_states(gs, o.state(), oracle.FASGD, f"{w.name} T={T} (sampled)")
            checks += 1
    g.srv.sync()
    return checks


def test_workload_25m_k8_full_stream_sampled():
    """P = 25M, lambda = 128, K = 8, Geometric(0.05) staleness: all 20,000
    pushes (2,500 fused passes, the benchmark's launch), checked every 200."""
    w = W["fasgd-25m-k8"]
    assert _sampled_stream(w, w.P, w.pushes, w.K) == w.pushes // 200


def test_workload_268m_k16_full_stream_sampled():
    """P = 2^28, lambda = 256, K = 16, Pareto(1.5) staleness, s_p up to 1: all
    2,000 pushes (125 passes), checked every 400.  A pool of 16 resident
    gradients (each batch uses every slot once)."""
    w = W["fasgd-268m-k16"]
    assert _sampled_stream(w, w.P, w.pushes, w.K, R=16) == w.pushes // 400


def test_bfasgd_full_stream():
    """B-FASGD at P = 200,003 over the workload's whole 10,000 pushes
    (lambda = 64, Poisson(8) staleness, ~20 % sent): each push selected with
    its client's v snapshot, every list bit-exact, the sparse apply's state
    within the bound every 100 pushes."""
    import torch
    w = W["bfasgd-25m"]
    P = 200_003
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    vsnap = [streams.client_v_snapshot(w, c, P) for c in range(w.lam)]
    c_push = calibrate_c(vsnap[0], 0.2)
    seed = 0xC0FFEE_1234_5678
    ps = streams.push_stream(w, w.pushes, 1)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=seed)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=seed)
    vsnap_t = [torch.from_numpy(v).cuda() for v in vsnap]
    idx = torch.empty(P, dtype=torch.int32, device="cuda")
    val = torch.empty(P, dtype=torch.float32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    sent = 0
    for t in range(w.pushes):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.select_compact(c, g.pool[s], idx, val, cnt, v=vsnap_t[c])
        oi, ov = o.srv.select_compact(c, pool[s], vsnap[c])
        m = int(cnt.item())
        assert m == oi.size, (t, m, oi.size)
        assert_bitwise(idx[:m].cpu().numpy(), oi, f"idx t={t}")
        assert_bitwise(val[:m].cpu().numpy(), ov, f"val t={t}")
        g.srv.push_sparse(c, j, idx, val, n_dev=cnt, n_max=P)
        g.srv.apply_pending(1)
        o.srv.push_sparse(c, j, oi, ov)
        o.srv.apply_pending(1)
        sent += m
        if (t + 1) % 100 == 0:
            compare_states(g.state(), o.state(), oracle.FASGD, f"bfasgd full stream T={t + 1}")
    g.srv.sync()
    assert 0.17 < sent / (P * w.pushes) < 0.23


def test_message_rule_full_stream():
    """The paper's literal per-message B-FASGD (Sec. 2.3) over the B-FASGD
    workload's whole 10,000-push stream (lambda = 64, Poisson(8) staleness)
    at P = 100,003: every decision equal to the oracle's, the state within
    the bound every 100 pushes."""
    import torch
    w = W["bfasgd-message-25m"].replace(R=8)
    P = 100_003
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    seed = 0x3E55A6E
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=40.0, seed=seed)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, c_push=40.0, seed=seed)
    ps = streams.push_stream(w, w.pushes, 1)
    flags = torch.full((w.pushes,), -1, dtype=torch.int32, device="cuda")
    for t in range(w.pushes):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.push_message(c, j, g.pool[s], sent_dev=flags[t:t + 1])
        g.srv.apply_pending(1)
        o.srv.push_message(c, j, pool[s])
        o.srv.apply_pending(1)
        if (t + 1) % 100 == 0:
            compare_states(g.state(), o.state(), oracle.FASGD, f"message stream T={t + 1}")
            got = flags[:t + 1].cpu().numpy()
            want = np.array(o.srv.message_log, dtype=np.int32)
            assert np.array_equal(got, want), f"decisions differ by T={t + 1}"
    assert 0 < int(flags.sum()) < w.pushes


def test_budget_rule_full_stream():
    """Per-tensor B-FASGD under a 20 % budget over the workload's whole
    10,000-push stream at P = 100,003 in 17 tensors (fast arithmetic): every
    push's decisions and count equal to the oracle's, its threshold within
    1e-5, the state within the bound every 100 pushes."""
    import torch
    w = W["bfasgd-tensor-25m"].replace(R=8)
    P = 100_003
    sizes = streams.tensor_sizes(5, P, 17)
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    seed = 0xB0D6E7
    g = CudaRun(w, oracle.FASGD, P, pool, th0, seed=seed)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, seed=seed)
    g.srv.set_tensors(sizes)
    o.srv.set_tensors(sizes)
    sent = torch.zeros(len(sizes), dtype=torch.uint8, device="cuda")
    cth = torch.zeros(1, dtype=torch.float32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    budget = P // 5
    ps = streams.push_stream(w, w.pushes, 1)
    for t in range(w.pushes):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.push_budget(c, j, g.pool[s], budget, sent, cth, cnt)
        g.srv.apply_pending(1)
        o.srv.push_budget(c, j, pool[s], budget)
        o.srv.apply_pending(1)
        osent, oc, om = o.srv.budget_log[-1]
        assert np.array_equal(sent.cpu().numpy(), osent), f"decisions differ at push {t}"
        assert int(cnt.item()) == om, t
        gc = float(cth.item())
        assert gc == oc or abs(gc - oc) <= 1e-5 * abs(oc), (t, gc, oc)
        if (t + 1) % 100 == 0:
            compare_states(g.state(), o.state(), oracle.FASGD, f"budget stream T={t + 1}")


def test_budget_rule_full_stream_exact_mode_bitwise():
    """The same per-tensor rule in exact arithmetic (fasgd_set_exact) over the
    whole 10,000-push stream at P = 300,007 in 160 tensors: v is then the
    same on both sides, so every push's tensor means, threshold c, decisions
    and count equal the oracle's bit for bit, and so does the final state."""
    import torch
    w = W["bfasgd-tensor-25m"].replace(R=8)
    P = 300_007
    sizes = streams.tensor_sizes(5, P, 160)
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    seed = 0xB0D6E7
    g = CudaRun(w, oracle.FASGD, P, pool, th0, seed=seed, exact=True)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, seed=seed)
    g.srv.set_tensors(sizes)
    o.srv.set_tensors(sizes)
    sent = torch.zeros(len(sizes), dtype=torch.uint8, device="cuda")
    cth = torch.zeros(1, dtype=torch.float32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    ps = streams.push_stream(w, w.pushes, 1)
    for t in range(w.pushes):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        g.srv.push_budget(c, j, g.pool[s], P // 5, sent, cth, cnt)
        g.srv.apply_pending(1)
        o.srv.push_budget(c, j, pool[s], P // 5)
        o.srv.apply_pending(1)
        osent, oc, om = o.srv.budget_log[-1]
        assert np.array_equal(sent.cpu().numpy(), osent), f"decisions differ at push {t}"
        assert int(cnt.item()) == om, t
        assert np.float32(cth.item()).view(np.uint32) == np.float32(oc).view(np.uint32), t
    compare_states(g.state(), o.state(), oracle.FASGD, "exact budget stream", exact=True)
