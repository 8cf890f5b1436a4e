"""Error codes of the C ABI with a live handle; a failed call changes nothing."""

import numpy as np
import pytest

import oracle
from gpu_util import CudaRun, assert_bitwise
from paper_1601_04033_gb300 import streams

pytestmark = pytest.mark.gpu


def _f():
    from paper_1601_04033_gb300 import fasgd
    return fasgd


def _snapshot(srv, P):
    import torch
    out = [torch.empty(P, device="cuda") for _ in range(4)]
    T = srv.get_state(*out) if srv.pending == 0 else None
    return [x.cpu().numpy() for x in out], T, srv.pending


def test_error_codes_leave_state_unchanged():
    import torch
    f = _f()
    P = 1001
    srv = f.Server(P, 4, 0.01, f.FASGD)
    srv.set_params(torch.linspace(-1, 1, P, device="cuda"))
    g = torch.ones(P + 8, device="cuda")
    srv.push(0, 0, g)
    srv.apply_pending(1)
    h = srv.h
    before, T0, _ = _snapshot(srv, P)
    checks = [
        (f.ERANGE, lambda: f.fasgd_push(h, 4, 0, g.data_ptr())),            # client == lambda
        (f.ERANGE, lambda: f.fasgd_push(h, -1, 0, g.data_ptr())),
        (f.ERANGE, lambda: f.fasgd_push(h, 0, T0 + 1, g.data_ptr())),      # j > T
        (f.ERANGE, lambda: f.fasgd_push(h, 0, -1, g.data_ptr())),
        (f.EINVAL, lambda: f.fasgd_push(h, 0, 0, None)),                    # NULL
        (f.EINVAL, lambda: f.fasgd_push(h, 0, 0, g.data_ptr() + 4)),        # misaligned
        (f.EAGAIN, lambda: f.fasgd_apply_pending(h, 1)),                    # nothing pending
        (f.EINVAL, lambda: f.fasgd_apply_pending(h, 0)),
        (f.EINVAL, lambda: f.fasgd_apply_pending(h, f.KMAX + 1)),
        (f.EINVAL, lambda: f.fasgd_set_hparams(h, 1.5, 0.9, 1e-4, 0, 0, 0)),
        (f.EINVAL, lambda: f.fasgd_set_hparams(h, 0.9, 1.0, 1e-4, 0, 0, 0)),
        (f.EINVAL, lambda: f.fasgd_set_hparams(h, 0.9, 0.9, -1.0, 0, 0, 0)),
        (f.EINVAL, lambda: f.fasgd_set_hparams(h, 0.9, 0.9, 1e-4, -1.0, 0, 0)),
        (f.EINVAL, lambda: f.fasgd_set_hparams(h, 0.9, 0.9, 1e-4, 0, float("nan"), 0)),
        (f.EINVAL, lambda: f.fasgd_push_sparse(h, 0, 0, None, None, None, 5)),
        (f.EINVAL, lambda: f.fasgd_push_sparse(h, 0, 0, g.data_ptr(), g.data_ptr(), None, P + 1)),
        (f.EINVAL, lambda: f.fasgd_push_sparse(h, 0, 0, g.data_ptr() + 2, g.data_ptr(), None, 3)),
        (f.ERANGE, lambda: f.bfasgd_select_compact(h, 9, g.data_ptr(), None, g.data_ptr(),
                                                    g.data_ptr(), g.data_ptr())),
        (f.EINVAL, lambda: f.bfasgd_select_compact(h, 0, g.data_ptr() + 4, None, g.data_ptr(),
                                                    g.data_ptr(), g.data_ptr())),
        (f.EINVAL, lambda: f.bfasgd_select_compact(h, 0, g.data_ptr(), None, None,
                                                    g.data_ptr(), g.data_ptr())),
        (f.EINVAL, lambda: f.fasgd_set_params(h, None)),
        (f.EINVAL, lambda: f.fasgd_set_state(h, None, None, None, None, -1)),
    ]
    for want, call in checks:
        rc = call()
        assert rc == want, (rc, want, f.fasgd_last_error(h))
        assert f.fasgd_last_error(h)
        assert srv.T == T0 and srv.pending == 0
    after, T1, _ = _snapshot(srv, P)
    for x, y in zip(before, after):
        assert_bitwise(x, y, "state after rejected calls")
    assert list(srv.push_counts()) == [0, 0, 0, 0]
    # Calls that need an empty queue refuse while pushes are pending.
    srv.push(1, 1, g)
    assert f.fasgd_set_stream(h, None) == f.EAGAIN
    assert f.fasgd_set_params(h, g.data_ptr()) == f.EAGAIN
    assert f.fasgd_get_state(h, None, None, None, None)[0] == f.EAGAIN
    assert f.fasgd_set_hparams(h, 0.9, 0.9, 1e-4, 0, 0, 0) == f.EAGAIN
    assert f.fasgd_apply_pending(h, 2) == f.EAGAIN and srv.pending == 1
    srv.apply_pending(1)
    srv.sync()
    srv.close()
    srv.close()


def test_host_push_and_pull_match_device_path():
    """fasgd_push_host (pinned host gradients, device staging) == fasgd_push."""
    import torch
    f = _f()
    w = streams.WORKLOADS["fasgd-1.29m"]
    P = 40_003
    pool = streams.gradient_pool(w, P, 8)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w.replace(R=8, K=4), 40, 4)
    a = CudaRun(w, oracle.FASGD, P, pool, th0)
    b = CudaRun(w, oracle.FASGD, P, pool, th0)
    host_pool = torch.from_numpy(pool).pin_memory()
    out = torch.empty(P, dtype=torch.float32).pin_memory()
    for k in range(10):
        cl, js, sl = ps.batch(k)
        a.push_batch(cl, js, sl)
        for c, j, s in zip(cl, js, sl):
            b.srv.push_host(int(c), int(j), host_pool[int(s)])
        b.srv.apply_pending(4)
        T = b.srv.pull(out)
        torch.cuda.current_stream().synchronize()
        assert T == 4 * (k + 1)
        assert_bitwise(out.numpy(), a.state()[0], f"pull after batch {k}")
    # At most KMAX host pushes may wait for an apply.
    for i in range(f.KMAX):
        b.srv.push_host(0, b.srv.T, host_pool[i % 8])
    with pytest.raises(f.FasgdError) as e:
        b.srv.push_host(0, b.srv.T, host_pool[0])
    assert e.value.code == f.EAGAIN
    b.srv.apply_pending(f.KMAX)
    b.srv.sync()


def test_a_pipeline_wait_that_never_completes_is_reported():
    """Failure detection without a fault: the dense pass's bounded pipeline
    waits, run on a barrier nothing completes, give up after about a second,
    raise flag 8, and fasgd_sync reports EDEVICE; the state is untouched and
    the handle keeps working."""
    import time
    import torch
    from paper_1601_04033_gb300 import fasgd
    P = 10_000
    srv = fasgd.Server(P, 2, 0.01, fasgd.FASGD)
    srv.set_params(torch.linspace(-1, 1, P, device="cuda"))
    g = torch.randn(P, device="cuda") * 0.01
    srv.push(0, 0, g)
    srv.apply_pending(1)
    srv.sync()
    before = [torch.empty(P, device="cuda") for _ in range(4)]
    srv.get_state(*before)
    launches = srv.launches
    t0 = time.time()
    srv.selftest_wait_expiry()
    with pytest.raises(fasgd.FasgdError) as e:
        srv.sync()
    took = time.time() - t0
    assert e.value.code == fasgd.EDEVICE
    assert "flags 0x8 " in str(e.value)      # only the pipeline-wait flag
    assert 0.9 < took < 60, took
    assert srv.launches == launches + 1
    after = [torch.empty(P, device="cuda") for _ in range(4)]
    srv.get_state(*after)
    for x, y in zip(before, after):
        assert torch.equal(x, y)
    srv.sync()                      # the flags were cleared
    srv.push(1, 1, g)               # and the handle still applies pushes
    srv.apply_pending(1)
    srv.sync()
    assert srv.T == 2
    srv.close()


@pytest.mark.parametrize("fail_at", [0, 1, 2, 3, 4])
def test_apply_pending_failing_partway_applies_each_push_once(fail_at):
    """Failure partway through a mixed batch, made on the host (the injected
    pass reports a launch failure and nothing runs for it): the call returns
    ECUDA, the pushes before the failed pass have left the queue and T has
    advanced by their number, the failed message or budget push keeps its
    draw counter; a retry of the rest then leaves the state bit for bit
    where one uninterrupted apply of the whole batch leaves it.  Passes of
    the batch: 0 two fused dense pushes, 1 a message push, 2 a sparse push,
    3 a budget push, 4 a dense push."""
    import torch
    from paper_1601_04033_gb300 import fasgd
    P, lam = 20_011, 4
    gen = torch.Generator(device="cuda").manual_seed(11)
    grads = [torch.randn(P, device="cuda", generator=gen) * 0.05 for _ in range(5)]
    idx = torch.arange(0, P, 3, dtype=torch.int32, device="cuda")
    val = grads[3][idx.long()].contiguous()
    theta0 = torch.randn(P, device="cuda", generator=gen) * 0.01

    def server():
        srv = fasgd.Server(P, lam, 0.01, fasgd.FASGD, c_push=3.0, seed=5)
        srv.set_params(theta0)
        srv.set_tensors([5000, 7011, 8000])
        return srv

    def queue(srv):
        srv.push(0, 0, grads[0])
        srv.push(1, 0, grads[1])
        srv.push_message(2, 0, grads[2])
        srv.push_sparse(3, 0, idx, val)
        srv.push_budget(1, 0, grads[4], 9000)
        srv.push(0, 0, grads[0])

    ref = server()
    queue(ref)
    ref.apply_pending(6)
    srv = server()
    queue(srv)
    pushes_before = [0, 2, 3, 4, 5][fail_at]     # pushes of the passes before the failed one
    srv.selftest_fail_pass(fail_at)
    with pytest.raises(fasgd.FasgdError) as e:
        srv.apply_pending(6)
    assert e.value.code == fasgd.ECUDA
    assert f"{pushes_before} of 6 pushes were applied" in str(e.value)
    assert srv.T == pushes_before and srv.pending == 6 - pushes_before
    counts = list(srv.push_counts())
    assert counts[2] == (1 if pushes_before > 2 else 0)      # the message push's draw
    assert counts[1] == (1 if pushes_before > 4 else 0)      # the budget push's draw
    srv.apply_pending(6 - pushes_before)
    srv.sync()
    ref.sync()
    assert srv.T == ref.T == 6 and srv.pending == 0
    assert list(srv.push_counts()) == list(ref.push_counts())
    a = [torch.empty(P, device="cuda") for _ in range(4)]
    b = [torch.empty(P, device="cuda") for _ in range(4)]
    srv.get_state(*a)
    ref.get_state(*b)
    for x, y, name in zip(a, b, ("theta", "n", "b", "v")):
        assert torch.equal(x, y), name
    srv.close()
    ref.close()


@pytest.mark.parametrize("variant,seed", [("FASGD", 1), ("FASGD", 2), ("FASGD", 3),
                                          ("SASGD", 4), ("ASGD", 5), ("FASGD_STD", 6)])
def test_random_protocol_against_oracle(variant, seed):
    """A random interleaving of every kind of call a server sees -- dense
    pushes from device and from pinned host memory, caller sparse lists,
    B-FASGD selects pushed as lists, per-message and per-tensor pushes,
    applies of random K (some with a launch failure injected partway and
    then retried), per-parameter, per-message and per-tensor fetches, and
    checkpoint round trips -- against the oracle driven the same way, in
    exact arithmetic, for each update rule: every list, decision and count bit
    for bit as it happens, and the state, timestamp and draw counters bit for
    bit at the end."""
    import torch
    from paper_1601_04033_gb300 import fasgd
    rng = np.random.default_rng(seed)
    P, lam, R = 12_007, 4, 6
    w = streams.WORKLOADS["bfasgd-tensor-25m"].replace(lam=lam, R=R)
    sizes = streams.tensor_sizes(seed, P, 7)
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    hp = (0.95, 0.95, 1e-4, 2.0, 1e-8, 77 + seed)
    alpha = 1e-5 if variant == "FASGD_STD" else 0.01   # the divide-by-std steps are ~1/std^2 larger
    srv = fasgd.Server(P, lam, alpha, getattr(fasgd, variant))
    srv.set_exact(True)
    srv.set_hparams(*hp)
    srv.set_fetch_threshold(1.5)
    srv.set_params(torch.from_numpy(th0).cuda())
    srv.set_tensors(sizes)
    o = oracle.OracleServer(P, lam, alpha, getattr(oracle, variant))
    o.set_hparams(*hp)
    o.set_fetch_threshold(1.5)
    o.set_params(th0)
    o.set_tensors(sizes)
    _, dpool = fasgd.aligned_vectors(pool)
    hpool = torch.from_numpy(pool).pin_memory()
    keep = []                                   # device lists borrowed until applied
    idx = torch.empty(P, dtype=torch.int32, device="cuda")
    val = torch.empty(P, dtype=torch.float32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    flag = torch.empty(1, dtype=torch.int32, device="cuda")
    sent = torch.zeros(len(sizes), dtype=torch.uint8, device="cuda")
    cdev = torch.zeros(1, dtype=torch.float32, device="cuda")
    kinds = ["dense", "host", "list", "select", "message", "budget", "apply", "apply",
             "fetch", "fetch_message", "fetch_budget", "checkpoint"]
    for step in range(400):
        kind = kinds[rng.integers(len(kinds))] if srv.pending < 20 else "apply"
        c = int(rng.integers(lam))
        T = srv.T
        assert T == o.T and srv.pending == len(o.fifo), step
        j = int(rng.integers(max(0, T - 5), T + 1))
        s = int(rng.integers(R))
        if kind == "dense":
            srv.push(c, j, dpool[s])
            o.push(c, j, pool[s])
        elif kind == "host":
            srv.push_host(c, j, hpool[s])
            o.push(c, j, pool[s])
        elif kind == "list":
            li = np.sort(rng.choice(P, int(rng.integers(0, P // 3)), replace=False)).astype(np.int32)
            lv = (rng.standard_normal(li.size) * 0.05).astype(np.float32)
            di, dv = torch.from_numpy(li).cuda(), torch.from_numpy(lv).cuda()
            keep.append((di, dv))
            srv.push_sparse(c, j, di, dv)
            o.push_sparse(c, j, li, lv)
        elif kind == "select":
            li, lv, lc = torch.empty_like(idx), torch.empty_like(val), torch.empty_like(cnt)
            keep.append((li, lv, lc))
            srv.select_compact(c, dpool[s], li, lv, lc)
            oi, ov = o.select_compact(c, pool[s])
            m = int(lc.item())
            assert m == oi.size, step
            assert_bitwise(li[:m].cpu().numpy(), oi, f"select idx {step}")
            assert_bitwise(lv[:m].cpu().numpy(), ov, f"select val {step}")
            srv.push_sparse(c, j, li, lv, n_dev=lc, n_max=P)
            o.push_sparse(c, j, oi, ov)
        elif kind == "message":
            srv.push_message(c, j, dpool[s])
            o.push_message(c, j, pool[s])
        elif kind == "budget":
            budget = int(rng.integers(0, P + 100))
            srv.push_budget(c, j, dpool[s], budget)
            o.push_budget(c, j, pool[s], budget)
        elif kind == "apply":
            if srv.pending == 0:
                continue
            K = int(rng.integers(1, min(srv.pending, 32) + 1))
            T0 = srv.T
            if rng.random() < 0.3:
                srv.selftest_fail_pass(int(rng.integers(0, 3)))
            try:
                srv.apply_pending(K)
            except fasgd.FasgdError as e:
                assert e.code == fasgd.ECUDA
                srv.selftest_fail_pass(-1)
                done = srv.T - T0
                assert srv.pending == len(o.fifo) - done
                srv.apply_pending(K - done)
            srv.selftest_fail_pass(-1)
            o.apply_pending(K)
        elif kind == "fetch":
            srv.fetch_compact(c, idx, val, cnt)
            oi, ov = o.fetch_compact(c)
            m = int(cnt.item())
            assert m == oi.size, step
            assert_bitwise(idx[:m].cpu().numpy(), oi, f"fetch idx {step}")
            assert_bitwise(val[:m].cpu().numpy(), ov, f"fetch val {step}")
        elif kind == "fetch_message":
            copy = torch.full((P,), 7.0, device="cuda")
            srv.fetch_message(c, copy, fetched_dev=flag)
            ocopy = np.full(P, 7.0, np.float32)
            ok = o.fetch_message(c, ocopy)
            assert int(flag.item()) == int(ok), step
            assert_bitwise(copy.cpu().numpy(), ocopy, f"fetched copy {step}")
        elif kind == "fetch_budget":
            budget = int(rng.integers(0, P + 100))
            copy = torch.full((P,), 7.0, device="cuda")
            srv.fetch_budget(c, copy, budget, sent_dev=sent, c_dev=cdev)
            ocopy = np.full(P, 7.0, np.float32)
            osent, oc, _ = o.fetch_budget(c, ocopy, budget)
            assert np.array_equal(sent.cpu().numpy(), osent), step
            assert np.float32(cdev.item()).view(np.uint32) == np.float32(oc).view(np.uint32), step
            assert_bitwise(copy.cpu().numpy(), ocopy, f"budget fetch copy {step}")
        elif kind == "checkpoint" and srv.pending == 0:
            st = [torch.empty(P, device="cuda") for _ in range(4)]
            Tc = srv.get_state(*st)
            srv.set_state(*st, Tc)
    while srv.pending:
        K = min(srv.pending, 32)
        srv.apply_pending(K)
        o.apply_pending(K)
    srv.sync()
    assert srv.T == o.T
    assert list(srv.push_counts()) == o.push_count
    assert list(srv.fetch_counts()) == o.fetch_count
    out = [torch.empty(P, device="cuda") for _ in range(4)]
    srv.get_state(*out)
    for x, y, name in zip(out, o.state()[:4], ("theta", "n", "b", "v")):
        assert_bitwise(x.cpu().numpy(), y.astype(np.float32), f"final {name}")
    srv.close()


def test_set_stream_orders_the_previous_streams_work():
    """fasgd_set_stream: a fused pass of 8 pushes at P = 25M enqueued on one
    stream, a switch to a second stream and a one-push pass enqueued there at
    once leave the state of the nine pushes applied in order -- bit for bit
    the state of the same calls on one stream.  (Were the second stream not
    ordered after the first, its pass would read theta, n, b, v while the
    first pass still writes them.)"""
    import torch
    from paper_1601_04033_gb300 import fasgd
    P, K = 25_000_000, 8
    gen = torch.Generator(device="cuda").manual_seed(11)
    grads = torch.randn(K + 1, P, device="cuda", generator=gen) * 0.01
    th0 = torch.randn(P, device="cuda", generator=gen) * 0.01
    torch.cuda.synchronize()

    def run(switch):
        first, second = torch.cuda.Stream(), torch.cuda.Stream()
        srv = fasgd.Server(P, 4, 0.001, fasgd.FASGD, stream=first)
        srv.set_params(th0)
        for k in range(K):
            srv.push(k % 4, 0, grads[k])
        srv.apply_pending(K)
        if switch:
            srv.set_stream(second)
        srv.push(0, K, grads[K])
        srv.apply_pending(1)
        srv.sync()
        out = [torch.empty(P, device="cuda") for _ in range(4)]
        assert srv.get_state(*out) == K + 1
        srv.close()
        return out

    for x, y in zip(run(False), run(True)):
        assert torch.equal(x, y)
