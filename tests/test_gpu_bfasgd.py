"""CUDA B-FASGD path (select / compact, sparse apply) against the oracle."""

import numpy as np
import pytest

import oracle
from gpu_util import (CudaRun, OracleRun, assert_bitwise, assert_close, compare_states)
from paper_1601_04033_gb300 import streams
from paper_1601_04033_gb300.calibrate import calibrate_c

pytestmark = pytest.mark.gpu

W = streams.WORKLOADS
SEED = 0xC0FFEE_1234_5678


def _select_gpu(srv, client, g_t, v_t=None):
    import torch
    P = g_t.numel()
    idx = torch.full((P,), -7, dtype=torch.int32, device="cuda")
    val = torch.full((P,), float("nan"), dtype=torch.float32, device="cuda")
    n = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    srv.select_compact(client, g_t, idx, val, n, v=v_t)
    m = int(n.item())
    return idx[:m].cpu().numpy(), val[:m].cpu().numpy(), m, (idx, val, n)


def _server(P, lam=8, c=1.0, variant=oracle.FASGD, seed=SEED):
    from paper_1601_04033_gb300 import fasgd
    return fasgd.Server(P, lam, 0.001, variant, c_push=c, eps_b=1e-8, seed=seed)


@pytest.mark.parametrize("P", [1, 3, 4, 5, 31, 33, 127, 128, 129, 1023, 8191, 8192, 8193,
                               16385, 100_003, 1_290_510])
def test_select_bit_exact(P):
    import torch
    rng = np.random.default_rng(P)
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)
    v = (10 ** rng.uniform(-1, 2, P)).astype(np.float32)
    g_t, v_t = torch.from_numpy(g).cuda(), torch.from_numpy(v).cuda()
    for c in (0.0, 0.5, calibrate_c(v, 0.2), 1e4, float("inf")):
        srv = _server(P, c=c)
        for push_no in range(2):
            client = 5
            gi, gv, m, _ = _select_gpu(srv, client, g_t, v_t)
            oi, ov = oracle.select(g, v, np.float32(c), 1e-8, SEED, client, push_no)
            assert m == oi.size, (P, c, push_no, m, oi.size)
            assert_bitwise(gi, oi, f"idx P={P} c={c}")
            assert_bitwise(gv, ov, f"val P={P} c={c}")
        assert list(srv.push_counts()) == [0, 0, 0, 0, 0, 2, 0, 0]
        srv.close()


def test_select_uses_live_v_when_v_is_null():
    import torch
    P = 50_000
    w = W["bfasgd-25m"]
    pool = streams.gradient_pool(w, P, 4)
    th0 = streams.theta0(w, P)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=2.0, seed=SEED)
    g.push_batch([0, 1], [0, 0], [0, 1])
    v_live = g.state()[3]
    gi, gv, m, _ = _select_gpu(g.srv, 3, g.pool[2])
    oi, ov = oracle.select(pool[2], v_live, 2.0, 1e-8, SEED, 3, 0)
    assert_bitwise(gi, oi, "idx")
    assert_bitwise(gv, ov, "val")


def _bfasgd_stream(P, n_pushes, w, c_target=0.2, check_every=100):
    """Select with each client's v snapshot, push the list, apply; both sides."""
    import torch
    lam = w.lam
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    vsnap = [streams.client_v_snapshot(w, c, P) for c in range(lam)]
    c_push = calibrate_c(vsnap[0], c_target)
    ps = streams.push_stream(w, n_pushes, 1)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    o = OracleRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    vsnap_t = [torch.from_numpy(v).cuda() for v in vsnap]
    sent = 0
    for t in range(n_pushes):
        cl, js, sl = ps.batch(t)
        c, j, s = int(cl[0]), int(js[0]), int(sl[0])
        gi, gv, m, bufs = _select_gpu(g.srv, c, g.pool[s], vsnap_t[c])
        oi, ov = o.srv.select_compact(c, pool[s], vsnap[c])
        assert m == oi.size
        assert_bitwise(gi, oi, f"idx t={t}")
        assert_bitwise(gv, ov, f"val t={t}")
        idx_t, val_t, n_t = bufs
        g.srv.push_sparse(c, j, idx_t, val_t, n_dev=n_t, n_max=P)
        g.srv.apply_pending(1)
        o.srv.push_sparse(c, j, oi, ov)
        o.srv.apply_pending(1)
        sent += m
        if (t + 1) % check_every == 0:
            compare_states(g.state(), o.state(), oracle.FASGD, f"bfasgd T={t + 1}")
    g.srv.sync()
    return sent / (P * n_pushes)


def test_bfasgd_stream_parity():
    w = W["bfasgd-25m"]
    frac = _bfasgd_stream(200_003, 300, w)
    assert 0.17 < frac < 0.23, frac


def test_bfasgd_c0_equals_dense_bitwise():
    import torch
    w = W["bfasgd-25m"]
    P = 77_777
    pool = streams.gradient_pool(w, P, 8)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w.replace(R=8), 40, 1)
    a = CudaRun(w, oracle.FASGD, P, pool, th0)
    b = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=0.0, seed=SEED)
    for t in range(40):
        cl, js, sl = ps.batch(t)
        a.push_batch(cl, js, sl)
        _, _, m, (idx, val, n) = _select_gpu(b.srv, int(cl[0]), b.pool[int(sl[0])])
        assert m == P
        b.srv.push_sparse(int(cl[0]), int(js[0]), idx, val, n_dev=n, n_max=P)
        b.srv.apply_pending(1)
    for x, y, name in zip(a.state()[:4], b.state()[:4], ("theta", "n", "b", "v")):
        assert_bitwise(x, y, name)


def test_empty_list_leaves_state():
    import torch
    w = W["bfasgd-25m"]
    P = 4099
    pool = streams.gradient_pool(w, P, 2)
    g = CudaRun(w, oracle.FASGD, P, pool, streams.theta0(w, P), c_push=float("inf"))
    g.push_batch([0], [0], [0])
    before = g.state()
    _, _, m, (idx, val, n) = _select_gpu(g.srv, 1, g.pool[1])
    assert m == 0
    g.srv.push_sparse(1, 1, idx, val, n_dev=n, n_max=P)
    g.srv.push_sparse(1, 1, idx, val, n_dev=None, n_max=0)
    g.srv.apply_pending(2)
    after = g.state()
    for x, y in zip(before[:4], after[:4]):
        assert_bitwise(x, y, "empty")
    assert after[4] == before[4] + 2
    g.srv.sync()


def test_device_flags_on_bad_lists():
    import torch
    from paper_1601_04033_gb300 import fasgd
    P = 1000
    srv = _server(P)
    srv.set_params(torch.zeros(P, device="cuda"))
    val = torch.ones(8, device="cuda")
    cases = [
        torch.tensor([1, 5, 1000, 7], dtype=torch.int32, device="cuda"),      # out of range
        torch.tensor([1, 5, -3, 9], dtype=torch.int32, device="cuda"),        # negative
        torch.tensor([1, 5, 5, 9], dtype=torch.int32, device="cuda"),         # not ascending
    ]
    for bad in cases:
        srv.push_sparse(0, srv.T, bad, val[:4])
        srv.apply_pending(1)
        with pytest.raises(fasgd.FasgdError) as e:
            srv.sync()
        assert e.value.code == fasgd.EDEVICE
        srv.sync()      # flags were cleared
    good = torch.tensor([0, 2, 4], dtype=torch.int32, device="cuda")
    over = torch.tensor([10], dtype=torch.int64, device="cuda")
    srv.push_sparse(0, srv.T, good, val[:3], n_dev=over, n_max=3)   # count above n_max
    srv.apply_pending(1)
    with pytest.raises(fasgd.FasgdError):
        srv.sync()
    srv.push_sparse(0, srv.T, good, val[:3])
    srv.apply_pending(1)
    srv.sync()


@pytest.mark.slow
def test_select_full_size_25m_bit_exact():
    import torch
    w = W["bfasgd-25m"]
    P = w.P
    g = streams.gradient_pool(w, P, 1)[0]
    v = streams.client_v_snapshot(w, 3, P)
    c = calibrate_c(v, 0.2)
    srv = _server(P, lam=w.lam, c=c)
    gi, gv, m, _ = _select_gpu(srv, 3, torch.from_numpy(g).cuda(), torch.from_numpy(v).cuda())
    oi, ov = oracle.select(g, v, c, 1e-8, SEED, 3, 0)
    assert m == oi.size and 0.19 < m / P < 0.21
    assert_bitwise(gi, oi, "idx 25M")
    assert_bitwise(gv, ov, "val 25M")


@pytest.mark.slow
def test_bfasgd_full_size_25m_sampled():
    """Select + sparse apply at P = 25M for 12 pushes; every list bit-exact,
    the state compared on sampled parameters."""
    import torch
    w = W["bfasgd-25m"].replace(R=4)
    P = w.P
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    vsnap = [streams.client_v_snapshot(w, c, P) for c in range(3)]
    c_push = calibrate_c(vsnap[0], 0.2)
    idx_s = streams.sample_indices(P, 20_000)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    o = OracleRun(w, oracle.FASGD, idx_s.size, np.ascontiguousarray(pool[:, idx_s]), th0[idx_s],
                  c_push=c_push, seed=SEED)
    pos = np.full(P, -1, np.int64)
    pos[idx_s] = np.arange(idx_s.size)
    counts = [0, 0, 0]
    for t in range(12):
        c, s, j = t % 3, t % 4, max(0, t - 2)
        gi, gv, m, (it, vt, nt) = _select_gpu(g.srv, c, g.pool[s], torch.from_numpy(vsnap[c]).cuda())
        oi, ov = oracle.select(pool[s], vsnap[c], c_push, 1e-8, SEED, c, counts[c])
        counts[c] += 1
        assert_bitwise(gi, oi, f"idx t={t}")
        assert_bitwise(gv, ov, f"val t={t}")
        g.srv.push_sparse(c, j, it, vt, n_dev=nt, n_max=P)
        g.srv.apply_pending(1)
        keep = pos[oi] >= 0
        o.srv.push_sparse(c, j, pos[oi[keep]].astype(np.int32), ov[keep])
        o.srv.apply_pending(1)
    g.srv.sync()
    gs = g.state()
    compare_states([x[idx_s] for x in gs[:4]] + [gs[4]], o.state(), oracle.FASGD, "bfasgd 25M")


@pytest.mark.slow
def test_bfasgd_full_size_2_28_sampled():
    """The bench's 2^28 exchange shape (bfasgd-268m): select with a client's v
    snapshot, then the sparse apply, for 4 pushes of 2 clients; every list
    bit-exact, the state compared on 20,000 sampled parameters."""
    import torch
    w = W["bfasgd-268m"].replace(R=2)
    P = w.P
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    vsnap = [streams.client_v_snapshot(w, c, P) for c in range(2)]
    c_push = calibrate_c(vsnap[0][:: P // (1 << 22)], 0.2)
    idx_s = streams.sample_indices(P, 20_000)
    g = CudaRun(w, oracle.FASGD, P, pool, th0, c_push=c_push, seed=SEED)
    o = OracleRun(w, oracle.FASGD, idx_s.size, np.ascontiguousarray(pool[:, idx_s]), th0[idx_s],
                  c_push=c_push, seed=SEED)
    pos = np.full(P, -1, np.int64)
    pos[idx_s] = np.arange(idx_s.size)
    counts = [0, 0]
    for t in range(4):
        c, s, j = t % 2, t % 2, max(0, t - 1)
        gi, gv, m, (it, vt, nt) = _select_gpu(g.srv, c, g.pool[s], torch.from_numpy(vsnap[c]).cuda())
        oi, ov = oracle.select(pool[s], vsnap[c], c_push, 1e-8, SEED, c, counts[c])
        counts[c] += 1
        assert 0.15 < m / P < 0.25
        assert_bitwise(gi, oi, f"idx t={t}")
        assert_bitwise(gv, ov, f"val t={t}")
        g.srv.push_sparse(c, j, it, vt, n_dev=nt, n_max=P)
        g.srv.apply_pending(1)
        keep = pos[oi] >= 0
        o.srv.push_sparse(c, j, pos[oi[keep]].astype(np.int32), ov[keep])
        o.srv.apply_pending(1)
    g.srv.sync()
    gs = g.state()
    compare_states([x[idx_s] for x in gs[:4]] + [gs[4]], o.state(), oracle.FASGD, "bfasgd 2^28")


@pytest.mark.slow
def test_select_max_p():
    """P = 2^31 - 1, the largest P int32 indices allow: c = 0 keeps every index
    (the last one is 2^31 - 2), c = inf keeps none, and at a 20% threshold every
    sampled parameter's membership matches the oracle's decision."""
    import torch
    P = (1 << 31) - 1
    gen = torch.Generator(device="cuda").manual_seed(1234)
    g_t = torch.randn(P, device="cuda", generator=gen)
    v_t = torch.empty(P, device="cuda").uniform_(1.0, 100.0, generator=gen)
    samp = streams.sample_indices(P, 4000)
    samp_t = torch.from_numpy(samp).cuda()
    g_s, v_s = g_t[samp_t].cpu().numpy(), v_t[samp_t].cpu().numpy()
    idx = torch.empty(P, dtype=torch.int32, device="cuda")
    val = torch.empty(P, dtype=torch.float32, device="cuda")
    n = torch.empty(1, dtype=torch.int64, device="cuda")
    for c in (0.0, float("inf"), 200.0):
        srv = _server(P, c=c)
        srv.select_compact(1, g_t, idx, val, n, v=v_t)
        m = int(n.item())
        if c == 0.0:
            assert m == P
            assert int(idx[-1].item()) == P - 1 and int(idx[0].item()) == 0
            assert bool((idx[samp_t] == samp_t.to(torch.int32)).all())
        elif c == float("inf"):
            assert m == 0
        else:
            kept = idx[:m]
            assert bool((kept[1:] > kept[:-1]).all())
            pos = torch.searchsorted(kept, samp_t.to(torch.int32))
            posc = pos.clamp(max=m - 1)
            member = (kept[posc] == samp_t.to(torch.int32)).cpu().numpy()
            vals = val[posc].cpu().numpy()
            for k, p in enumerate(samp):
                u = oracle.draw(SEED, 1, 0, int(p))
                want = oracle.decide(u, float(v_s[k]), c, 1e-8)
                assert bool(member[k]) == want, (p, member[k], want)
                if want:
                    assert np.float32(vals[k]).view(np.uint32) == np.float32(g_s[k]).view(np.uint32)
        srv.close()
        del srv


def test_select_at_the_threshold_bit_exact():
    """Every parameter's v is set so that its Eq. 9 threshold falls within an
    ulp of its own draw u_p (computed by the oracle): the decisions then hinge
    on the exact comparison, which both sides must take identically."""
    import torch
    P = 40_000
    c = 3.0
    eps_b = 0.0
    seed, client, push_no = 0xABCDEF, 2, 0
    u = np.array([oracle.draw(seed, client, push_no, p) for p in range(P)], dtype=np.float64)
    u = np.clip(u, 1, 2 ** 24 - 2)
    # a / (a + c) = u / 2^24  <=>  a = c u / (2^24 - u); nudge by -1, 0, +1 ulp.
    a = (c * u / (2.0 ** 24 - u)).astype(np.float32)
    nudge = np.random.default_rng(7).integers(-1, 2, P)
    a = np.nextafter(a, np.where(nudge > 0, np.inf, -np.inf).astype(np.float32)).astype(np.float32)
    a = np.where(nudge == 0, (c * u / (2.0 ** 24 - u)).astype(np.float32), a)
    v = a.astype(np.float32)
    g = np.random.default_rng(8).standard_normal(P).astype(np.float32)
    srv = _server(P, c=c, seed=seed)
    srv.set_hparams(0.95, 0.95, 1e-4, c, eps_b, seed)
    gi, gv, m, _ = _select_gpu(srv, client, torch.from_numpy(g).cuda(), torch.from_numpy(v).cuda())
    oi, ov = oracle.select(g, v, c, eps_b, seed, client, push_no)
    assert 0.2 * P < m < 0.8 * P          # the decisions really are split
    assert_bitwise(gi, oi, "idx at threshold")
    assert_bitwise(gv, ov, "val at threshold")


def test_select_threshold_over_the_whole_fp32_range():
    """The exact Eq. 9 test away from ordinary magnitudes: thresholds placed at
    each parameter's own draw (within an ulp) for c from subnormal to 2^110,
    on both sides of the c = 2^79 switch between the kernel's two scalings,
    and a above 2^104 (where a * 2^24 leaves the fp32 range) with small c,
    where every parameter is sent.  Bit-exact against the oracle."""
    import torch
    P = 40_000
    eps_b = 0.0
    seed, client = 0xABCDEF, 3
    u = np.array([oracle.draw(seed, client, 0, p) for p in range(P)], dtype=np.float64)
    u = np.clip(u, 1, 2 ** 24 - 2)
    nudge = np.random.default_rng(17).integers(-1, 2, P)
    g = np.random.default_rng(18).standard_normal(P).astype(np.float32)
    g_t = torch.from_numpy(g).cuda()
    cases = []
    for c in (2.0 ** -140, 2.0 ** -100, 3.0, 2.0 ** 78, 2.0 ** 79, 2.0 ** 80, 2.0 ** 110):
        with np.errstate(over="ignore", under="ignore"):
            a = np.minimum(c * u / (2.0 ** 24 - u), 3.0e38).astype(np.float32)
        up = np.nextafter(a, np.float32(np.inf))
        down = np.nextafter(a, np.float32(0))
        v = np.where(nudge > 0, up, np.where(nudge < 0, down, a)).astype(np.float32)
        cases.append((c, v, True))
    big = (2.0 ** np.random.default_rng(19).uniform(104, 127.9, P)).astype(np.float32)
    for c in (0.0, 1.0, 2.0 ** 78):
        cases.append((c, big, False))
    for k, (c, v, split) in enumerate(cases):
        c32 = float(np.float32(c))
        srv = _server(P, c=c32, seed=seed)
        srv.set_hparams(0.95, 0.95, 1e-4, c32, eps_b, seed)
        gi, gv, m, _ = _select_gpu(srv, client, g_t, torch.from_numpy(v).cuda())
        oi, ov = oracle.select(g, v, c32, eps_b, seed, client, 0)
        if split:
            assert 0.1 * P < m < 0.9 * P, (c, m)
        else:
            assert m == P, (c, m)
        assert_bitwise(gi, oi, f"idx c={c}")
        assert_bitwise(gv, ov, f"val c={c}")
        srv.close()


def test_sparse_apply_divide_by_std_matches_dense_at_c0():
    import torch
    w = W["bfasgd-25m"]
    P = 20_011
    pool = streams.gradient_pool(w, P, 4)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w.replace(R=4), 25, 1)
    a = CudaRun(w, oracle.FASGD_STD, P, pool, th0)
    b = CudaRun(w, oracle.FASGD_STD, P, pool, th0, c_push=0.0, seed=SEED)
    o = OracleRun(w, oracle.FASGD_STD, P, pool, th0)
    for t in range(25):
        cl, js, sl = ps.batch(t)
        a.push_batch(cl, js, sl)
        o.push_batch(cl, js, sl)
        _, _, m, (idx, val, n) = _select_gpu(b.srv, int(cl[0]), b.pool[int(sl[0])])
        b.srv.push_sparse(int(cl[0]), int(js[0]), idx, val, n_dev=n, n_max=P)
        b.srv.apply_pending(1)
    for x, y, name in zip(a.state()[:4], b.state()[:4], ("theta", "n", "b", "v")):
        assert_bitwise(x, y, name)
    compare_states(a.state(), o.state(), oracle.FASGD_STD, "std variant")


def _mid_sizes():
    """About 5M parameters (~600 tiles of 8,192): a whole number of tiles,
    partial last tiles of 1 and 4,099 parameters, one short of a tile
    boundary, and a size whose tile count is no multiple of the SM count."""
    at = 608 * 8192
    return [at - 1, at, at + 1, at + 4099, at + 97 * 8192 + 12_345]


@pytest.mark.parametrize("which", range(5))
def test_select_mid_sizes_bit_exact(which):
    """Push and fetch selects at about 5M parameters against the oracle, for
    thresholds in both forms of the Eq. 9 test (c below and above 2^79) and two
    calls of each stream."""
    import torch
    P = _mid_sizes()[which]
    rng = np.random.default_rng(P)
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)
    for lo, hi, cs in ((-1, 2, (0.0, 5.0, float("inf"))), (28, 34, (1e30,))):
        v = (10 ** rng.uniform(lo, hi, P)).astype(np.float32)
        g_t, v_t = torch.from_numpy(g).cuda(), torch.from_numpy(v).cuda()
        for c in cs:
            srv = _server(P, c=c)
            srv.set_fetch_threshold(c)
            srv.set_params(g_t)             # fetches compact theta = g
            for call in range(2):
                gi, gv, m, _ = _select_gpu(srv, 5, g_t, v_t)
                oi, ov = oracle.select(g, v, np.float32(c), 1e-8, SEED, 5, call)
                assert m == oi.size, (P, c, call, m, oi.size)
                if 0.0 < c < float("inf"):
                    assert 0 < m < P
                assert_bitwise(gi, oi, f"push idx P={P} c={c}")
                assert_bitwise(gv, ov, f"push val P={P} c={c}")
                idx = torch.empty(P, dtype=torch.int32, device="cuda")
                val = torch.empty(P, dtype=torch.float32, device="cuda")
                n = torch.empty(1, dtype=torch.int64, device="cuda")
                srv.fetch_compact(5, idx, val, n, v=v_t)
                fm = int(n.item())
                fi, fv = oracle.fetch_select(g, v, np.float32(c), 1e-8, SEED, 5, call)
                assert fm == fi.size, (P, c, call, fm, fi.size)
                assert_bitwise(idx[:fm].cpu().numpy(), fi, f"fetch idx P={P} c={c}")
                assert_bitwise(val[:fm].cpu().numpy(), fv, f"fetch val P={P} c={c}")
            srv.sync()
            srv.close()
