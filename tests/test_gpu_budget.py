"""CUDA path of per-tensor B-FASGD under a bandwidth budget (tensor means,
budget threshold, per-tensor Eq. 9 decisions, ranged apply and fetch copy)
against the oracle."""

import numpy as np
import pytest

import oracle
from gpu_util import HP, assert_bitwise, assert_close, binding, compare_states, torch_cuda
from paper_1601_04033_gb300 import streams

pytestmark = pytest.mark.gpu

SEED = 0xB0D6E7


class Pair:
    """A CUDA server and the oracle server on the same partition and inputs."""

    def __init__(self, P, sizes, lam=4, variant=oracle.FASGD, exact=False, eps_b=1e-8,
                 pool_workload="bfasgd-tensor-25m", R=8, alpha=None):
        torch = torch_cuda()
        f = binding()
        w = streams.WORKLOADS[pool_workload].replace(lam=lam, R=R)
        if alpha is not None:
            w = w.replace(alpha=alpha)
        self.w, self.P, self.variant, self.exact = w, P, variant, exact
        self.pool = streams.gradient_pool(w, P)
        th0 = streams.theta0(w, P)
        self.srv = f.Server(P, lam, w.alpha, variant, gamma=HP["gamma"], beta=HP["beta"],
                            eps=HP["eps"], eps_b=eps_b, seed=SEED)
        self.srv.set_exact(exact)
        self._buf, self.dpool = f.aligned_vectors(self.pool)
        self.srv.set_params(torch.from_numpy(th0).cuda())
        self.srv.set_tensors(sizes)
        self.o = oracle.OracleServer(P, lam, w.alpha, variant, gamma=HP["gamma"],
                                     beta=HP["beta"], eps=HP["eps"], eps_b=eps_b, seed=SEED)
        self.o.set_params(th0)
        self.o.set_tensors(sizes)
        self.T = len(sizes)
        self.sent = torch.zeros(self.T, dtype=torch.uint8, device="cuda")
        self.c = torch.zeros(1, dtype=torch.float32, device="cuda")
        self.count = torch.zeros(1, dtype=torch.int64, device="cuda")

    def push(self, client, j, slot, budget):
        self.srv.push_budget(client, j, self.dpool[slot], budget, self.sent, self.c, self.count)
        self.srv.apply_pending(1)
        self.o.push_budget(client, j, self.pool[slot], budget)
        self.o.apply_pending(1)
        return self.decision(), self.o.budget_log[-1]

    def decision(self):
        return (self.sent.cpu().numpy(), float(self.c.item()), int(self.count.item()))

    def check_decision(self, got, want, where, c_exact=True):
        gs, gc, gm = got
        ws, wc, wm = want
        assert np.array_equal(gs, ws), f"{where}: decisions differ at {np.flatnonzero(gs != ws)}"
        assert gm == wm, f"{where}: count {gm} vs {wm}"
        if c_exact:
            assert np.float32(gc).view(np.uint32) == np.float32(wc).view(np.uint32), \
                f"{where}: c {gc!r} vs {wc!r}"
        else:
            assert gc == wc or abs(gc - wc) <= 1e-5 * abs(wc), f"{where}: c {gc!r} vs {wc!r}"

    def gpu_state(self):
        torch = torch_cuda()
        out = [torch.empty(self.P, dtype=torch.float32, device="cuda") for _ in range(4)]
        T = self.srv.get_state(*out)
        return [x.cpu().numpy() for x in out] + [T]


def _stream(pair, n, frac, check_every):
    ps = streams.push_stream(pair.w, n, 1)
    budget = int(frac * pair.P)
    total = 0
    for t in range(n):
        cl, js, sl = ps.batch(t)
        got, want = pair.push(int(cl[0]), int(js[0]), int(sl[0]), budget)
        pair.check_decision(got, want, f"push {t}", c_exact=pair.exact)
        total += got[2]
        if (t + 1) % check_every == 0:
            compare_states(pair.gpu_state(), list(pair.o.state()), pair.variant,
                           f"budget T={t + 1}", exact=pair.exact)
    return total


@pytest.mark.parametrize("P,T", [(7_850, 2), (100_003, 17), (1_290_510, 160)])
def test_budget_stream_exact_mode_bitwise(P, T):
    """Exact arithmetic: every decision, threshold and count equal, state bit
    for bit (v is the same on both sides, so every tensor mean is too)."""
    pair = Pair(P, streams.tensor_sizes(3, P, T), exact=True)
    n = 200 if P < 1_000_000 else 60
    total = _stream(pair, n, 0.2, 20)
    assert 0 < total < n * P


@pytest.mark.parametrize("P,T,variant", [(100_003, 17, oracle.FASGD),
                                          (65_537, 33, oracle.FASGD_STD),
                                          (65_537, 33, oracle.SASGD)])
def test_budget_stream_fast_arithmetic(P, T, variant):
    """Default arithmetic: decisions equal, threshold within 1e-5, state within
    the dense bound (n and b bitwise)."""
    kw = {"alpha": 1e-6} if variant == oracle.FASGD_STD else {}
    pair = Pair(P, streams.tensor_sizes(5, P, T), variant=variant, **kw)
    _stream(pair, 200, 0.3, 100)


def test_decisions_at_a_fixed_state_many_budgets():
    """Fetch decisions (no state change) at one shared server state for a
    sweep of budgets: threshold, decisions, counts and copies exactly equal."""
    torch = torch_cuda()
    P, T = 300_007, 150
    sizes = streams.tensor_sizes(9, P, T)
    pair = Pair(P, sizes)
    rng = np.random.default_rng(4)
    # Per-tensor scales so the allocation has something to follow.
    scale = np.repeat(10 ** rng.uniform(-1, 2, T), sizes).astype(np.float32)
    v = (scale * rng.uniform(0.5, 1.5, P)).astype(np.float32)
    theta = (rng.standard_normal(P) * 0.01).astype(np.float32)
    z = np.zeros(P, np.float32)
    pair.srv.set_state(*[torch.from_numpy(x).cuda() for x in (theta, z, z, v)], 3)
    pair.o.theta[:], pair.o.v[:], pair.o.T = theta, v, 3
    for k, budget in enumerate([0, 1, 17, 1000, P // 10, P // 3, P // 2, P - 1, P, 2 * P]):
        copy = torch.full((P,), 9.0, device="cuda")
        pair.srv.fetch_budget(k % 4, copy, budget, pair.sent, pair.c, pair.count)
        ocopy = np.full(P, 9.0, np.float32)
        want = pair.o.fetch_budget(k % 4, ocopy, budget)
        pair.check_decision(pair.decision(), want, f"budget {budget}")
        assert_bitwise(copy.cpu().numpy(), ocopy, f"fetched copy, budget {budget}")
        if budget >= P:
            assert want[1] == 0.0 and want[2] == P
    assert list(pair.srv.fetch_counts()) == pair.o.fetch_count


@pytest.mark.parametrize("T", [2, 33, 600, 3000])
def test_thresholds_jumping_between_calls(T):
    """Budgets in shuffled order on one stream, tensor means spread over twelve
    decades: the threshold jumps far between calls and E is far from linear
    over the first brackets, so the search leans on its even-split fallback.
    Every threshold and decision equals the oracle's (2, 33, 600 and 3000
    tensors give 31, 7, 3 and 1 candidates per round)."""
    torch = torch_cuda()
    P = 200_003
    sizes = streams.tensor_sizes(11, P, T)
    pair = Pair(P, sizes)
    rng = np.random.default_rng(T)
    scale = np.repeat(10 ** rng.uniform(-6, 6, T), sizes).astype(np.float32)
    v = (scale * rng.uniform(0.9, 1.1, P)).astype(np.float32)
    z = np.zeros(P, np.float32)
    pair.srv.set_state(*[torch.from_numpy(x).cuda() for x in (z, z, z, v)], 5)
    pair.o.theta[:], pair.o.v[:], pair.o.T = z, v, 5
    budgets = [P // 2, 3, P - 7, P // 50, 0, P // 5, 1, P // 3, 2 * P, P // 7, 100, P // 2]
    for k, budget in enumerate(budgets):
        copy = torch.zeros(P, device="cuda")
        pair.srv.fetch_budget(1, copy, budget, pair.sent, pair.c, pair.count)
        want = pair.o.fetch_budget(1, np.zeros(P, np.float32), budget)
        pair.check_decision(pair.decision(), want, f"T={T} call {k} budget {budget}")


def test_full_budget_is_the_dense_pass_bitwise():
    """budget >= P transmits every tensor (c = 0): the same bits as fasgd_push."""
    torch = torch_cuda()
    f = binding()
    P = 200_003
    sizes = streams.tensor_sizes(2, P, 40)
    pair = Pair(P, sizes)
    dense = f.Server(P, 4, pair.w.alpha, f.FASGD, gamma=HP["gamma"], beta=HP["beta"],
                     eps=HP["eps"], eps_b=1e-8, seed=SEED)
    dense.set_params(torch.from_numpy(streams.theta0(pair.w, P)).cuda())
    ps = streams.push_stream(pair.w, 30, 1)
    for t in range(30):
        cl, js, sl = ps.batch(t)
        pair.srv.push_budget(int(cl[0]), int(js[0]), pair.dpool[int(sl[0])], P)
        pair.srv.apply_pending(1)
        dense.push(int(cl[0]), int(js[0]), pair.dpool[int(sl[0])])
        dense.apply_pending(1)
    out = [torch.empty(P, device="cuda") for _ in range(4)]
    dense.get_state(*out)
    for x, y, name in zip(pair.gpu_state()[:4], out, ("theta", "n", "b", "v")):
        assert_bitwise(x, y.cpu().numpy(), name)
    # The item sums are formed once; afterwards the apply keeps them current.
    assert pair.srv.launches == 1 + 30 * 2


def test_zero_budget_and_zero_statistics():
    """With eps_b = 0 and v = 0 at the start no tensor is ever sent (a_t = 0);
    a zero budget sends (almost) nothing."""
    P = 20_011
    sizes = streams.tensor_sizes(1, P, 9)
    pair = Pair(P, sizes, eps_b=0.0)
    ps = streams.push_stream(pair.w, 10, 1)
    for t in range(10):
        cl, js, sl = ps.batch(t)
        got, want = pair.push(int(cl[0]), int(js[0]), int(sl[0]), P // 2)
        pair.check_decision(got, want, f"zero stats push {t}")
        assert got[2] == 0 and got[1] == 0.0
    compare_states(pair.gpu_state(), list(pair.o.state()), oracle.FASGD, "zero stats")
    pair = Pair(P, sizes)
    for t in range(10):
        cl, js, sl = ps.batch(t)
        pair.push(int(cl[0]), int(js[0]), int(sl[0]), P)   # fills v
    for t in range(10):
        cl, js, sl = ps.batch(t)
        got, want = pair.push(int(cl[0]), int(js[0]), int(sl[0]), 0)
        pair.check_decision(got, want, f"zero budget push {t}", c_exact=False)
    compare_states(pair.gpu_state(), list(pair.o.state()), oracle.FASGD, "zero budget")


def test_item_sums_follow_every_change_of_v():
    """Budget pushes interleaved with dense, sparse and per-message pushes and a
    state restore (all of which rewrite v): every decision still equals the
    oracle's, which forms the tensor means from scratch each time."""
    torch = torch_cuda()
    P = 90_001
    sizes = streams.tensor_sizes(4, P, 23)
    pair = Pair(P, sizes, exact=True)
    pair.srv.set_hparams(HP["gamma"], HP["beta"], HP["eps"], 3.0, 1e-8, SEED)
    pair.o.set_hparams(HP["gamma"], HP["beta"], HP["eps"], 3.0, 1e-8, SEED)
    ps = streams.push_stream(pair.w, 60, 1)
    idx = torch.empty(P, dtype=torch.int32, device="cuda")
    val = torch.empty(P, dtype=torch.float32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    mid = mid_o = None
    for t in range(60):
        cl, js, sl = ps.batch(t)
        c, j, slot = int(cl[0]), int(js[0]), int(sl[0])
        kind = t % 5
        if kind == 1:
            pair.srv.push(c, j, pair.dpool[slot])
            pair.srv.apply_pending(1)
            pair.o.push(c, j, pair.pool[slot])
            pair.o.apply_pending(1)
        elif kind == 2:
            pair.srv.select_compact(c, pair.dpool[slot], idx, val, cnt)
            pair.srv.push_sparse(c, j, idx, val, n_dev=cnt, n_max=P)
            pair.srv.apply_pending(1)
            oi, ov = pair.o.select_compact(c, pair.pool[slot])
            pair.o.push_sparse(c, j, oi, ov)
            pair.o.apply_pending(1)
        elif kind == 3:
            pair.srv.push_message(c, j, pair.dpool[slot])
            pair.srv.apply_pending(1)
            pair.o.push_message(c, j, pair.pool[slot])
            pair.o.apply_pending(1)
        else:
            got, want = pair.push(c, j, slot, P // 4)
            pair.check_decision(got, want, f"interleaved push {t}")
        if t == 30:
            mid = pair.gpu_state()
            mid_o = [x.copy() for x in pair.o.state()[:4]]
        if t == 45:
            # Restore the state of T = 31 on both sides (v changes behind the sums).
            pair.srv.set_state(*[torch.from_numpy(x).cuda() for x in mid[:4]], pair.srv.T)
            pair.o.theta[:], pair.o.n[:], pair.o.b[:], pair.o.v[:] = mid_o
    compare_states(pair.gpu_state(), list(pair.o.state()), oracle.FASGD, "interleaved",
                   exact=True)


@pytest.mark.parametrize("sizes", [
    [1] * 64 + [70_000],                        # one-parameter tensors, one multi-item tensor
    [3, 5, 40_001, 7, 16_384, 16_385, 2],       # item cuts at and around the chunk size
    [100_003],                                  # one tensor: the per-message statistic
])
def test_ragged_partitions(sizes):
    P = int(sum(sizes))
    pair = Pair(P, np.array(sizes), exact=True)
    _stream(pair, 40, 0.4, 10)


@pytest.mark.parametrize("sizes", [[1], [1, 1, 1], [2, 3], [5], [1, 1, 1, 1, 1]])
def test_tiny_partitions(sizes):
    """A handful of parameters, one-parameter tensors, no whole 16-byte quad."""
    P = int(sum(sizes))
    pair = Pair(P, np.array(sizes), exact=True)
    _stream(pair, 30, 0.5, 10)


def test_maximum_tensor_count():
    f = binding()
    P = 50_000
    sizes = streams.tensor_sizes(11, P, f.BFASGD_TMAX)
    pair = Pair(P, sizes, exact=True)
    _stream(pair, 20, 0.25, 10)


def test_errors():
    torch = torch_cuda()
    f = binding()
    srv = f.Server(1000, 2, 0.01, f.FASGD)
    g = torch.zeros(1000, device="cuda")
    with pytest.raises(f.FasgdError) as e:
        srv.push_budget(0, 0, g, 10)                    # no partition
    assert e.value.code == f.EINVAL
    for bad in ([500, 499], [1000, 0], [0, 1000], [1] * (f.BFASGD_TMAX + 1)):
        with pytest.raises(f.FasgdError) as e:
            srv.set_tensors(bad)
        assert e.value.code == f.EINVAL
    srv.set_tensors([400, 600])
    with pytest.raises(f.FasgdError) as e:
        srv.push_budget(0, 0, g, -1)
    assert e.value.code == f.EINVAL
    with pytest.raises(f.FasgdError) as e:
        srv.push_budget(2, 0, g, 10)
    assert e.value.code == f.ERANGE
    srv.push_budget(0, 0, g, 10)
    with pytest.raises(f.FasgdError) as e:
        srv.set_tensors([1000])                         # pushes pending
    assert e.value.code == f.EAGAIN
    srv.apply_pending(1)
    srv.sync()


@pytest.mark.slow
def test_full_size_25m_160_tensors():
    """P = 25,000,000 in 160 tensors, the launch configuration the benchmark
    times: 12 pushes at a 20 % budget and 12 fetches at 10 %; decisions and
    counts exact, thresholds within 1e-5, the state on sampled parameters."""
    torch = torch_cuda()
    w = streams.WORKLOADS["bfasgd-tensor-25m"]
    P = w.P
    sizes = streams.tensor_sizes(w.seed, P, w.tensors)
    pair = Pair(P, sizes, pool_workload=w.name, R=4)
    ps = streams.push_stream(pair.w, 12, 1)
    for t in range(12):
        cl, js, sl = ps.batch(t)
        got, want = pair.push(int(cl[0]), int(js[0]), int(sl[0]), int(0.2 * P))
        pair.check_decision(got, want, f"25M push {t}", c_exact=False)
        copy = torch.zeros(P, device="cuda")
        pair.srv.fetch_budget(t % 4, copy, int(0.1 * P), pair.sent, pair.c, pair.count)
        fgot = pair.decision()
        ocopy = np.zeros(P, np.float32)
        fwant = pair.o.fetch_budget(t % 4, ocopy, int(0.1 * P))
        pair.check_decision(fgot, fwant, f"25M fetch {t}", c_exact=False)
        idx = streams.sample_indices(P, 20_000, seed=t)
        assert_close(copy.cpu().numpy()[idx], ocopy[idx], "25M fetched copy")
    gs = pair.gpu_state()
    idx = streams.sample_indices(P, 50_000)
    os_ = pair.o.state()
    compare_states([x[idx] for x in gs[:4]] + [gs[4]], [x[idx] for x in os_[:4]] + [os_[4]],
                   oracle.FASGD, "25M sampled")


@pytest.mark.slow
def test_size_2_28_64_tensors():
    """P = 2^28 in 64 tensors (work items of 32,768 parameters, ~8,200 items):
    three pushes at a 20 % budget and three fetches at 10 %, decisions and
    counts exact, thresholds within 1e-5, the state on sampled parameters."""
    torch = torch_cuda()
    P = 1 << 28
    sizes = streams.tensor_sizes(4, P, 64)
    pair = Pair(P, sizes, pool_workload="fasgd-268m-k16", R=4)
    ps = streams.push_stream(pair.w, 3, 1)
    for t in range(3):
        cl, js, sl = ps.batch(t)
        got, want = pair.push(int(cl[0]), int(js[0]), int(sl[0]), int(0.2 * P))
        pair.check_decision(got, want, f"2^28 push {t}", c_exact=False)
        copy = torch.zeros(P, device="cuda")
        pair.srv.fetch_budget(t % 4, copy, int(0.1 * P), pair.sent, pair.c, pair.count)
        ocopy = np.zeros(P, np.float32)
        fwant = pair.o.fetch_budget(t % 4, ocopy, int(0.1 * P))
        pair.check_decision(pair.decision(), fwant, f"2^28 fetch {t}", c_exact=False)
        idx = streams.sample_indices(P, 20_000, seed=t)
        assert_close(copy.cpu().numpy()[idx], ocopy[idx], "2^28 fetched copy")
        del copy
    idx = torch.from_numpy(streams.sample_indices(P, 50_000)).cuda()
    full = [torch.empty(P, device="cuda") for _ in range(4)]
    T = pair.srv.get_state(*full)
    gs = [x[idx].cpu().numpy() for x in full] + [T]
    del full
    ih = idx.cpu().numpy()
    os_ = pair.o.state()
    compare_states(gs, [x[ih] for x in os_[:4]] + [os_[4]], oracle.FASGD, "2^28 sampled")


@pytest.mark.slow
def test_largest_size_and_tensor_count():
    """P = 2^31 - 1 in BFASGD_TMAX tensors (work items of 262,144 parameters,
    the largest decision block): with v constant on each tensor the tensor
    means are exact, so the oracle's threshold, decisions and counts are
    computed from the partition alone and must match the GPU's bit for bit;
    the fetched copy holds theta exactly on the transmitted tensors."""
    torch = torch_cuda()
    f = binding()
    P = (1 << 31) - 1
    T = f.BFASGD_TMAX
    sizes = streams.tensor_sizes(13, P, T)
    rng = np.random.default_rng(13)
    vt = np.float32(2.0) ** rng.integers(-6, 7, T).astype(np.float32)   # exact means
    srv = f.Server(P, 2, 0.001, f.FASGD, eps_b=1e-8, seed=SEED)
    srv.set_tensors(sizes)
    size_t = torch.from_numpy(sizes).cuda()
    v = torch.repeat_interleave(torch.from_numpy(vt).cuda(), size_t, output_size=P)
    theta = torch.arange(P, device="cuda", dtype=torch.float32)
    z = torch.zeros(P, device="cuda")
    srv.set_state(theta, z, z, v, 0)
    del v, z
    sent = torch.zeros(T, dtype=torch.uint8, device="cuda")
    c = torch.zeros(1, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int64, device="cuda")
    copy = torch.full((P,), -1.0, device="cuda")
    off = np.concatenate([[0], np.cumsum(sizes)])
    for k, budget in enumerate([P, P // 5, 0]):
        srv.fetch_budget(1, copy, budget, sent, c, cnt)
        want_c = oracle.budget_c(sizes, vt, 1e-8, budget)
        want_sent, want_m = oracle.tensor_select(sizes, vt, want_c, 1e-8, SEED, 1, 1, k)
        assert np.float32(c.item()).view(np.uint32) == np.float32(want_c).view(np.uint32), (budget, c.item(), want_c)
        assert np.array_equal(sent.cpu().numpy(), want_sent), budget
        assert int(cnt.item()) == want_m
        if budget == P:
            assert want_m == P
        # The copy equals theta on a sample of parameters of every transmitted tensor.
        for t in np.flatnonzero(want_sent)[:64]:
            for p in (int(off[t]), int(off[t + 1]) - 1, int((off[t] + off[t + 1]) // 2)):
                assert copy[p].item() == theta[p].item(), (budget, t, p)


def test_mixed_kinds_in_one_apply():
    """Dense, per-tensor, sparse and per-message pushes queued together and
    applied by single fasgd_apply_pending calls: each in arrival order at its
    own timestamp, bit for bit with the oracle (exact mode)."""
    torch = torch_cuda()
    P = 40_009
    sizes = streams.tensor_sizes(6, P, 11)
    pair = Pair(P, sizes, exact=True)
    pair.srv.set_hparams(HP["gamma"], HP["beta"], HP["eps"], 2.0, 1e-8, SEED)
    pair.o.set_hparams(HP["gamma"], HP["beta"], HP["eps"], 2.0, 1e-8, SEED)
    idx = torch.empty(P, dtype=torch.int32, device="cuda")
    val = torch.empty(P, dtype=torch.float32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    for rnd in range(6):
        T = pair.srv.T
        assert T == pair.o.T
        s0, s1, s2, s3, s4 = [(rnd * 5 + k) % 8 for k in range(5)]
        pair.srv.push(0, T, pair.dpool[s0])
        pair.o.push(0, T, pair.pool[s0])
        pair.srv.push_budget(1, max(T - 1, 0), pair.dpool[s1], P // 3, pair.sent, pair.c, pair.count)
        pair.o.push_budget(1, max(T - 1, 0), pair.pool[s1], P // 3)
        pair.srv.select_compact(2, pair.dpool[s2], idx, val, cnt)
        pair.srv.push_sparse(2, T, idx, val, n_dev=cnt, n_max=P)
        oi, ov = pair.o.select_compact(2, pair.pool[s2])
        pair.o.push_sparse(2, T, oi, ov)
        pair.srv.push_message(3, T, pair.dpool[s3])
        pair.o.push_message(3, T, pair.pool[s3])
        pair.srv.push(0, T, pair.dpool[s4])
        pair.o.push(0, T, pair.pool[s4])
        pair.srv.apply_pending(5)
        pair.o.apply_pending(5)
        pair.check_decision(pair.decision(), pair.o.budget_log[-1], f"mixed round {rnd}")
    compare_states(pair.gpu_state(), list(pair.o.state()), oracle.FASGD, "mixed", exact=True)
