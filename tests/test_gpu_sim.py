"""The closed-loop simulation on the CUDA path against the oracle's: the
gradient and loss kernels, and whole runs (dispatcher, stale clients, server
pass, refresh) for every update rule and fetch mode."""

import numpy as np
import pytest

import oracle
import oracle.sim as osim
from gpu_util import assert_bitwise, assert_close
from paper_1601_04033_gb300 import streams

pytestmark = pytest.mark.gpu


def _f():
    from paper_1601_04033_gb300 import fasgd
    return fasgd


@pytest.mark.parametrize("P", [1, 3, 4, 5, 1023, 65_537])
def test_sim_grad_and_loss_kernels(P):
    import torch
    f = _f()
    h, star, sigma = streams.quadratic_objective(7, P)
    th = (np.random.default_rng(P).standard_normal(P) * 0.1).astype(np.float32)
    _, (dth, dh, dst, dsg, dg) = f.aligned_vectors(np.stack([th, h, star, sigma, th]))
    stream = torch.cuda.current_stream().cuda_stream
    for client, n in ((0, 0), (3, 17), (5, 1 << 33)):
        rc = f.fasgd_sim_quadratic_grad(P, dth.data_ptr(), dh.data_ptr(), dst.data_ptr(),
                                        dsg.data_ptr(), 1234, client, n, dg.data_ptr(), stream)
        assert rc == f.OK
        want = oracle.sim_grad(th, h, star, sigma, 1234, client, n)
        assert_bitwise(dg.cpu().numpy(), want, f"sim grad P={P} client={client}")
    scratch = torch.empty(1024, dtype=torch.float64, device="cuda")
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    assert f.fasgd_sim_quadratic_loss(P, dth.data_ptr(), dh.data_ptr(), dst.data_ptr(),
                                      scratch.data_ptr(), loss.data_ptr(), stream) == f.OK
    want = oracle.sim_loss(th, h, star)
    assert abs(float(loss.item()) - want) <= 1e-10 * want


RULES = [oracle.ASGD, oracle.SASGD, oracle.FASGD, oracle.FASGD_STD]


@pytest.mark.parametrize("exact", [False, True])
@pytest.mark.parametrize("variant", RULES)
@pytest.mark.parametrize("K,fetch", [(1, "full"), (4, "full"), (1, "param"), (1, "message")])
def test_simulation_against_oracle(variant, K, fetch, exact):
    """Whole closed-loop runs.  In exact mode every run reproduces the oracle
    bit for bit.  With the fast forms (default) the loss curves agree to 1e-5;
    the parameters are compared only in exact mode, because the loop feeds the
    server's few-ulp differences back through the clients' copies, and
    parameters near the stability limit amplify them (ASGD / SASGD are exact
    in both modes and are compared bit for bit)."""
    from paper_1601_04033_gb300.sim import Simulation
    P, lam, n_batches = 20_011, 8, 120
    alpha = {oracle.ASGD: 0.02, oracle.SASGD: 0.1, oracle.FASGD: 0.002,
             oracle.FASGD_STD: 2e-5}[variant]
    obj = streams.quadratic_objective(3, P)
    th0 = np.zeros(P, np.float32)
    sched = streams.dispatch_schedule(3, lam, n_batches, K, rho=0.5)
    c_fetch = {"full": 0.0, "param": 30.0, "message": 30.0}[fetch]
    g = Simulation(P, lam, alpha, variant, K=K, seed=9, fetch=fetch, c_fetch=c_fetch,
                   objective=obj, theta0=th0, exact=exact)
    o = osim.OracleSimulation(P, lam, alpha, variant, seed=9, fetch=fetch, c_fetch=c_fetch,
                              objective=obj, theta0=th0)
    gl = g.run(sched, log_every=40)
    ol = o.run(sched, log_every=40)
    assert gl.shape == ol.shape
    np.testing.assert_allclose(gl, ol, rtol=1e-10 if exact else 1e-5)
    th = g.torch.empty(P, device="cuda")
    g.srv.pull(th)
    if exact or variant in (oracle.ASGD, oracle.SASGD):
        assert_bitwise(th.cpu().numpy(), o.srv.theta.astype(np.float32), "sim theta")
    if fetch == "full":
        assert gl[-1] < gl[0]
    g.close()


@pytest.mark.parametrize("exact", [False, True])
@pytest.mark.parametrize("variant", [oracle.FASGD, oracle.SASGD])
@pytest.mark.parametrize("mode", ["fetch", "push", "both"])
def test_simulation_with_per_tensor_budgets(variant, mode, exact):
    """Closed loop with per-tensor budgets: fetches of 10 % of P, pushes of
    30 % of P, or both, over 12 tensors whose curvature scales differ.  Exact
    mode reproduces the oracle bit for bit; the fast forms agree in loss."""
    from paper_1601_04033_gb300.sim import Simulation
    P, lam, n_batches = 20_011, 8, 120
    alpha = {oracle.SASGD: 0.005, oracle.FASGD: 0.0005}[variant]   # curvatures up to ~100
    sizes = streams.tensor_sizes(7, P, 12)
    obj = streams.quadratic_objective(3, P, tensors=sizes)
    th0 = np.zeros(P, np.float32)
    sched = streams.dispatch_schedule(3, lam, n_batches, 1, rho=0.5)
    kw = dict(seed=9, objective=obj, theta0=th0, eps_b=1e-3, tensor_sizes=sizes,
              fetch="budget" if mode in ("fetch", "both") else "full",
              fetch_budget=P // 10, push_budget=(3 * P // 10) if mode in ("push", "both") else None)
    g = Simulation(P, lam, alpha, variant, exact=exact, **kw)
    o = osim.OracleSimulation(P, lam, alpha, variant, **kw)
    gl = g.run(sched, log_every=40)
    ol = o.run(sched, log_every=40)
    np.testing.assert_allclose(gl, ol, rtol=1e-10 if exact else 1e-5)
    if exact or variant == oracle.SASGD:
        th = g.torch.empty(P, device="cuda")
        g.srv.pull(th)
        assert_bitwise(th.cpu().numpy(), o.srv.theta.astype(np.float32), "budget sim theta")
    if variant == oracle.SASGD:
        assert gl[-1] < gl[0]
    moved = int(g.fetched_params.item()) + int(g.pushed_params.item())
    assert 0 < moved < n_batches * P * (2 if mode == "both" else 1)
    g.close()

