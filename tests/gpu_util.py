"""Helpers shared by the GPU parity tests: drive the CUDA path (through the
C ABI binding) and the CPU oracle on the same seeded stream, and compare."""

from __future__ import annotations

import math

import numpy as np

import oracle
from paper_1601_04033_gb300 import streams

# Tolerance for fp32 parameters and statistics against the oracle, per
# element: |gpu - oracle| <= RTOL * |oracle| + ATOL.
RTOL = 1e-5
ATOL = 1e-7

HP = dict(gamma=0.95, beta=0.95, eps=1e-4, eps_b=1e-8)


def torch_cuda():
    import torch
    return torch


def binding():
    from paper_1601_04033_gb300 import fasgd
    return fasgd


def assert_close(gpu, ora, what):
    gpu = np.asarray(gpu, dtype=np.float64)
    ora = np.asarray(ora, dtype=np.float64)
    with np.errstate(invalid="ignore"):
        d = np.abs(gpu - ora)
    bound = RTOL * np.abs(ora) + ATOL
    bad = np.nonzero(~((d <= bound) | (gpu == ora)))[0]   # equal infinities match
    if bad.size:
        i = bad[np.argmax((d[bad] - bound[bad]))]
        raise AssertionError(f"{what}: {bad.size} of {gpu.size} outside tolerance; worst at {i}: "
                             f"gpu={gpu[i]!r} oracle={ora[i]!r} |d|={d[i]:.3e} bound={bound[i]:.3e}")


def assert_bitwise(gpu, ora, what):
    g = np.ascontiguousarray(gpu)
    o = np.ascontiguousarray(ora)
    assert g.dtype == o.dtype and g.shape == o.shape, (what, g.dtype, o.dtype, g.shape, o.shape)
    if g.dtype == np.float32:
        g, o = g.view(np.uint32), o.view(np.uint32)
    bad = np.nonzero(g != o)[0]
    assert bad.size == 0, f"{what}: {bad.size} elements differ, first at {bad[:5]}"


class CudaRun:
    """A CUDA-path server fed from a device-resident gradient pool."""

    def __init__(self, w: streams.Workload, variant: int, P: int, pool: np.ndarray,
                 theta0: np.ndarray, **hp):
        torch = torch_cuda()
        f = binding()
        h = dict(HP)
        h.update(hp)
        self.srv = f.Server(P, w.lam, w.alpha, variant, gamma=h["gamma"], beta=h["beta"],
                            eps=h["eps"], c_push=h.get("c_push", 0.0), eps_b=h["eps_b"],
                            seed=h.get("seed", 0))
        self.srv.set_exact(bool(h.get("exact", False)))
        self.P = P
        self._pool_buf, self.pool = f.aligned_vectors(pool)
        self.srv.set_params(torch.from_numpy(theta0).cuda())

    def push_batch(self, clients, js, slots):
        for c, j, s in zip(clients, js, slots):
            self.srv.push(int(c), int(j), self.pool[int(s)])
        self.srv.apply_pending(len(clients))

    def state(self):
        torch = torch_cuda()
        out = [torch.empty(self.P, dtype=torch.float32, device="cuda") for _ in range(4)]
        T = self.srv.get_state(*out)
        return [x.cpu().numpy() for x in out] + [T]


class OracleRun:
    def __init__(self, w: streams.Workload, variant: int, P: int, pool: np.ndarray,
                 theta0: np.ndarray, real: str = "f32", **hp):
        h = dict(HP)
        h.update(hp)
        self.srv = oracle.OracleServer(P, w.lam, w.alpha, variant, real=real,
                                       gamma=h["gamma"], beta=h["beta"], eps=h["eps"],
                                       c_push=h.get("c_push", 0.0), eps_b=h["eps_b"],
                                       seed=h.get("seed", 0))
        h.pop("exact", None)
        self.srv.set_params(theta0)
        self.pool = pool

    def push_batch(self, clients, js, slots):
        for c, j, s in zip(clients, js, slots):
            self.srv.push(int(c), int(j), self.pool[int(s)])
        self.srv.apply_pending(len(clients))

    def state(self):
        return list(self.srv.state())


def compare_states(gs, os_, variant, where, exact=False):
    names = ("theta", "n", "b", "v")
    assert gs[4] == os_[4], f"{where}: timestamps differ {gs[4]} vs {os_[4]}"
    if variant in (oracle.ASGD, oracle.SASGD):
        assert_bitwise(gs[0], os_[0].astype(np.float32), f"{where} theta")
        return
    if exact:   # exact arithmetic mode: every array bit for bit
        for k in range(4):
            assert_bitwise(gs[k], os_[k].astype(np.float32), f"{where} {names[k]}")
        return
    # n and b are formed with the same once-rounded fp32 sequence on both sides.
    assert_bitwise(gs[1], os_[1].astype(np.float32), f"{where} n")
    assert_bitwise(gs[2], os_[2].astype(np.float32), f"{where} b")
    for k in (0, 3):
        assert_close(gs[k], os_[k], f"{where} {names[k]}")


def run_parity(w, variant, P, n_pushes, K, check_every=None, real="f32", **hp):
    """Run GPU and oracle in lockstep; compare at every T multiple of lcm(100, K)."""
    check_every = check_every or (100 * K // math.gcd(100, K))
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w, n_pushes, K)
    g = CudaRun(w, variant, P, pool, th0, **hp)
    o = OracleRun(w, variant, P, pool, th0, real=real, **hp)
    checks = 0
    for b in range(n_pushes // K):
        cl, js, sl = ps.batch(b)
        g.push_batch(cl, js, sl)
        o.push_batch(cl, js, sl)
        T = (b + 1) * K
        if T % check_every == 0:
            compare_states(g.state(), o.state(), variant, f"{w.name} var={variant} P={P} K={K} T={T}",
                           exact=bool(hp.get("exact", False)))
            checks += 1
    assert checks > 0
    return g, o


def ring_P(extra: int = 500_017) -> int:
    """A parameter count the bulk-copy ring (not the plain-grid pass) handles
    on this GPU: 8 tiles of 2048 per SM, plus a ragged remainder."""
    torch = torch_cuda()
    return 8 * torch.cuda.get_device_properties(0).multi_processor_count * 2048 + extra


def run_parity_sampled(w, variant, P, n_pushes, K, count=20_000, **hp):
    """Like run_parity, but the oracle runs on `count` sampled parameters only
    (the update is elementwise, so that sub-problem is exact); compared at
    every T multiple of lcm(100, K)."""
    torch = torch_cuda()
    every = 100 * K // math.gcd(100, K)
    pool = streams.gradient_pool(w, P)
    th0 = streams.theta0(w, P)
    ps = streams.push_stream(w, n_pushes, K)
    idx = streams.sample_indices(P, count)
    g = CudaRun(w, variant, P, pool, th0, **hp)
    o = OracleRun(w, variant, idx.size, np.ascontiguousarray(pool[:, idx]), th0[idx], **hp)
    del pool
    idx_t = torch.from_numpy(idx).cuda()
    full = [torch.empty(P, device="cuda") for _ in range(4)]
    checks = 0
    for b in range(n_pushes // K):
        batch = ps.batch(b)
        g.push_batch(*batch)
        o.push_batch(*batch)
        if ((b + 1) * K) % every == 0:
            T = g.srv.get_state(*full)
            gs = [x[idx_t].cpu().numpy() for x in full] + [T]
            compare_states(gs, o.state(), variant, f"{w.name} var={variant} P={P} K={K} T={T} "
                           "(sampled)", exact=bool(hp.get("exact", False)))
            checks += 1
    assert checks > 0
    g.srv.sync()
    return checks
