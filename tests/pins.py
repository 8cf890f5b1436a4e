"""Checks that pin the CPU oracle to what the paper and the mathematics fix.

Each ``check_*`` takes an ``Libs`` (the fp32 and fp64 oracle builds) and
raises AssertionError on a mismatch.  ``test_oracle_pins.py`` runs them on
the real oracle; ``test_oracle_mutants.py`` runs them on copies of the oracle
with a planted mistake and requires that at least one fails.

None of these re-types the oracle's recursion: the references are closed
forms, the unrolled (non-recursive) series, hand-worked values, exact
rational arithmetic, published known-answer vectors, numpy's own fp32 SGD
step, and invariants between the variants.
"""

from __future__ import annotations

import dataclasses
import json
import math
import os
from fractions import Fraction

import numpy as np

import oracle
from oracle import ASGD, FASGD, FASGD_STD, SASGD

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@dataclasses.dataclass
class Libs:
    f32: object
    f64: object

    def lib(self, real):
        return self.f32 if real == "f32" else self.f64


def real_libs() -> Libs:
    return Libs(oracle._load("f32"), oracle._load("f64"))


def _server(libs, real, P, variant, alpha=0.25, lam=4, **hp):
    return oracle.OracleServer(P, lam, alpha, variant, real=real, lib=libs.lib(real), **hp)


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-300))


# --------------------------------------------------------------------------
# Hand trace exact in binary (Eq. 4-8)
# --------------------------------------------------------------------------
def check_hand_trace(libs: Libs):
    gold = json.load(open(os.path.join(GOLDEN, "hand_trace_fasgd.json")))
    hp = gold["hparams"]
    env = {"sqrt": math.sqrt}
    for real in ("f32", "f64"):
        s = _server(libs, real, 1, FASGD, alpha=hp["alpha"], gamma=hp["gamma"],
                    beta=hp["beta"], eps=hp["eps"])
        s.set_params(np.array([hp["theta0"]]))
        g = np.array([hp["g"]], dtype=np.float32)
        for k, st in enumerate(gold["steps"]):
            s.push(0, s.T, g)          # tau = 0
            s.apply_pending(1)
            want = {key: eval(st[key], env) for key in ("n", "b", "v", "theta")}
            got = {"n": s.n[0], "b": s.b[0], "v": s.v[0], "theta": s.theta[0]}
            for key in want:
                if st["exact_in_binary"]:
                    assert float(got[key]) == want[key], (real, k, key, got[key], want[key])
                else:
                    tol = 4e-7 if real == "f32" else 1e-15
                    assert abs(float(got[key]) - want[key]) <= tol * abs(want[key]), \
                        (real, k, key, got[key], want[key])


# --------------------------------------------------------------------------
# Constant gradient: closed-form geometric series (Eq. 4-8)
# --------------------------------------------------------------------------
def check_std_variant_closed_form(libs: Libs):
    """Divide-by-std reading: under a constant gradient, v averages
    sqrt(gamma^k (1 - gamma^k) g^2 + eps) and theta moves by coef g / v."""
    gvals = np.array([0.8, -0.25, 3e-3, 0.0], dtype=np.float32)
    P = gvals.shape[0]
    gamma, beta, eps, alpha = 0.9, 0.85, 1e-4, 0.02
    theta0 = np.array([0.01, -0.02, 0.0, 0.03], np.float32)
    for real, steps, tol in (("f32", 30, 2e-5), ("f64", 50, 1e-11)):
        s = _server(libs, real, P, FASGD_STD, alpha=alpha, gamma=gamma, beta=beta, eps=eps)
        s.set_params(theta0)
        G, B = float(np.float32(gamma)), float(np.float32(beta))
        E, A = float(np.float32(eps)), float(np.float32(alpha))
        g64 = gvals.astype(np.float64)
        theta_ref = theta0.astype(np.float64).copy()
        stds = []
        for i in range(1, steps + 1):
            s.push(0, s.T, gvals)
            s.apply_pending(1)
            gi = G ** i
            stds.append(np.sqrt(gi * (1 - gi) * g64 ** 2 + E))
            v_ref = (1 - B) * sum(B ** (i - k) * stds[k - 1] for k in range(1, i + 1))
            theta_ref = theta_ref - A * g64 / v_ref
            assert _rel(s.v, v_ref) <= tol, (real, i, "v")
            assert np.max(np.abs(s.theta - theta_ref)) <= tol * (np.max(np.abs(theta_ref)) + 1e-3)
    # The two readings differ (v is an average of std in one, of 1/std in the other).
    a = _server(libs, "f32", P, FASGD)
    b = _server(libs, "f32", P, FASGD_STD)
    for s in (a, b):
        s.push(0, 0, gvals)
        s.apply_pending(1)
    assert not np.array_equal(a.v, b.v)


def check_constant_gradient_closed_form(libs: Libs):
    gvals = np.array([1.0, -0.5, 0.03125, -2e-3, 0.3, 7e-5, -1.25, 0.0], dtype=np.float32)
    P = gvals.shape[0]
    gamma, beta, eps, alpha = 0.9, 0.8, 1e-4, 0.01
    rng = np.random.default_rng(5)
    taus = rng.integers(0, 6, 60)
    theta0 = np.linspace(-0.02, 0.02, P).astype(np.float32)
    for real, steps, tol in (("f32", 40, 2e-5), ("f64", 60, 1e-11)):
        s = _server(libs, real, P, FASGD, alpha=alpha, gamma=gamma, beta=beta, eps=eps)
        s.set_params(theta0)
        G, B = float(np.float32(gamma)), float(np.float32(beta))
        E, A = float(np.float32(eps)), float(np.float32(alpha))
        g64 = gvals.astype(np.float64)
        theta_ref = theta0.astype(np.float64).copy()
        rs = []
        for i in range(1, steps + 1):
            tau = min(int(taus[i - 1]), s.T)     # j = T - tau must be >= 0
            s.push(0, s.T - tau, gvals)
            s.apply_pending(1)
            gi = G ** i
            n_ref = (1 - gi) * g64 ** 2
            b_ref = (1 - gi) * g64
            var_ref = gi * (1 - gi) * g64 ** 2
            rs.append(1 / np.sqrt(var_ref + E))
            v_ref = (1 - B) * sum(B ** (i - k) * rs[k - 1] for k in range(1, i + 1))
            theta_ref = theta_ref - A / max(tau, 1) * g64 / v_ref
            assert _rel(s.n, n_ref) <= tol, (real, i, "n")
            assert _rel(s.b, b_ref) <= tol, (real, i, "b")
            assert _rel(s.v, v_ref) <= tol, (real, i, "v")
            assert np.max(np.abs(s.theta - theta_ref)) <= tol * (np.max(np.abs(theta_ref)) + 1e-3), \
                (real, i, "theta")


# --------------------------------------------------------------------------
# Random gradients, mixed staleness, dense and sparse pushes: the unrolled
# series form of Eq. 4-8 (and Eq. 1-2) evaluated directly in fp64.
# --------------------------------------------------------------------------
def _series_reference(variant, theta0, events, alpha, gamma, beta, eps):
    """events: list of (tau, {p: g}) in arrival order.  Returns theta, n, b, v."""
    P = theta0.shape[0]
    th = theta0.astype(np.float64).copy()
    n = np.zeros(P)
    b = np.zeros(P)
    v = np.zeros(P)
    for p in range(P):
        hist = [(tau, g[p]) for tau, g in events if p in g]
        rs = []
        step_sum = 0.0
        for i in range(1, len(hist) + 1):
            tau_i, g_i = hist[i - 1]
            c_i = alpha if variant == ASGD else alpha / max(tau_i, 1)
            if variant in (FASGD, FASGD_STD):
                n_i = sum((1 - gamma) * gamma ** (i - k) * hist[k - 1][1] ** 2 for k in range(1, i + 1))
                b_i = sum((1 - gamma) * gamma ** (i - k) * hist[k - 1][1] for k in range(1, i + 1))
                std = math.sqrt(max(n_i - b_i ** 2, 0.0) + eps)
                rs.append(1 / std if variant == FASGD else std)
                v_i = sum((1 - beta) * beta ** (i - k) * rs[k - 1] for k in range(1, i + 1))
                step_sum += c_i * g_i / v_i
                n[p], b[p], v[p] = n_i, b_i, v_i
            else:
                step_sum += c_i * g_i
        th[p] = float(theta0[p]) - step_sum
    return th, n, b, v


def check_series_bruteforce(libs: Libs):
    rng = np.random.default_rng(11)
    P = 7
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    gamma, beta, eps, alpha = 0.85, 0.7, 1e-3, 0.05
    steps = 24
    plan = []
    T = 0
    for t in range(steps):
        g = (rng.standard_normal(P) * rng.choice([0.01, 0.3, 1.0])).astype(np.float32)
        d = int(rng.integers(0, 5))
        j = T - min(d, T)
        if t % 3 == 2:      # a sparse push on a random ascending subset
            idx = np.sort(rng.choice(P, int(rng.integers(0, P + 1)), replace=False)).astype(np.int32)
            plan.append(("sparse", j, idx, g[idx]))
        else:
            plan.append(("dense", j, None, g))
        T += 1
    for variant in (ASGD, SASGD, FASGD, FASGD_STD):
        events = []
        for T, (kind, j, idx, g) in enumerate(plan):
            tau = T - j
            if kind == "dense":
                events.append((tau, {p: float(g[p]) for p in range(P)}))
            else:
                events.append((tau, {int(p): float(x) for p, x in zip(idx, g)}))
        G, B = float(np.float32(gamma)), float(np.float32(beta))
        E, A = float(np.float32(eps)), float(np.float32(alpha))
        ref = _series_reference(variant, theta0, events, A, G, B, E)
        for real, tol in (("f32", 3e-5), ("f64", 1e-12)):
            s = _server(libs, real, P, variant, alpha=alpha, gamma=gamma, beta=beta, eps=eps)
            s.set_params(theta0)
            for kind, j, idx, g in plan:
                if kind == "dense":
                    s.push(1, j, g)
                else:
                    s.push_sparse(1, j, idx, g)
                s.apply_pending(1)
            got = s.state()[:4]
            for name, a, r in zip(("theta", "n", "b", "v"), got, ref):
                # elementwise relative error, floored at tol * the array's scale
                bound = tol * (np.abs(r) + np.max(np.abs(r)) + 1e-30)
                assert np.all(np.abs(a - r) <= bound), (variant, real, name,
                                                        np.max(np.abs(a - r) / bound) * tol)


# --------------------------------------------------------------------------
# Variant invariants (Eq. 1-2 vs plain SGD; SASGD vs ASGD)
# --------------------------------------------------------------------------
def check_variant_invariants(libs: Libs):
    rng = np.random.default_rng(3)
    P = 33
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    grads = [(rng.standard_normal(P) * 0.1).astype(np.float32) for _ in range(12)]
    alpha = 0.0123
    # tau = 0 for every push: ASGD == SASGD == plain fp32 SGD (numpy), bitwise.
    outs = {}
    for variant in (ASGD, SASGD):
        s = _server(libs, "f32", P, variant, alpha=alpha)
        s.set_params(theta0)
        for g in grads:
            s.push(0, s.T, g)
            s.apply_pending(1)
        outs[variant] = s.theta.copy()
    sgd = theta0.copy()
    a32 = np.float32(alpha)
    for g in grads:
        sgd = (sgd - a32 * g).astype(np.float32)
    assert np.array_equal(outs[ASGD].view(np.uint32), sgd.view(np.uint32))
    assert np.array_equal(outs[SASGD].view(np.uint32), sgd.view(np.uint32))
    # Constant tau = 3: SASGD(alpha) == ASGD(fl(alpha / 3)), bitwise.
    tau = 3
    s1 = _server(libs, "f32", P, SASGD, alpha=alpha)
    s2 = _server(libs, "f32", P, ASGD, alpha=float(np.float32(np.float32(alpha) / np.float64(tau))))
    for s in (s1, s2):
        s.set_params(theta0)
        for _ in range(tau):        # advance T so that j = T - 3 is legal
            s.push(0, s.T, np.zeros(P, np.float32))
            s.apply_pending(1)
    th_start = s1.theta.copy()
    assert np.array_equal(s2.theta, th_start)
    for g in grads:
        for s in (s1, s2):
            s.push(0, s.T - tau, g)
            s.apply_pending(1)
    assert np.array_equal(s1.theta.view(np.uint32), s2.theta.view(np.uint32))
    # SASGD with tau = 0 and tau = 1 coincide (the max(tau, 1) reading).
    assert oracle.coef(SASGD, alpha, 0, lib=libs.f32) == oracle.coef(SASGD, alpha, 1, lib=libs.f32)
    assert oracle.coef(ASGD, alpha, 7, lib=libs.f32) == np.float32(alpha)
    # The statistics never move under ASGD / SASGD.
    for variant in (ASGD, SASGD):
        s = _server(libs, "f32", P, variant, alpha=alpha)
        s.push(0, 0, grads[0])
        s.apply_pending(1)
        assert not s.n.any() and not s.b.any() and not s.v.any()


def check_dense_equals_full_sparse(libs: Libs):
    rng = np.random.default_rng(4)
    P = 40
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    full = np.arange(P, dtype=np.int32)
    for variant in (ASGD, SASGD, FASGD):
        a = _server(libs, "f32", P, variant)
        c = _server(libs, "f32", P, variant)
        a.set_params(theta0)
        c.set_params(theta0)
        for t in range(15):
            g = (rng.standard_normal(P) * 0.2).astype(np.float32)
            j = a.T - min(t % 4, a.T)
            a.push(t % 4, j, g)
            c.push_sparse(t % 4, j, full, g)
            a.apply_pending(1)
            c.apply_pending(1)
        for x, y in zip(a.state()[:4], c.state()[:4]):
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32))


# --------------------------------------------------------------------------
# Eq. 9: the fp32 send decision against exact rational arithmetic
# --------------------------------------------------------------------------
def _exact_decide(u, v, c, eps_b):
    with np.errstate(over="ignore"):
        a = np.float32(np.float32(v) + np.float32(eps_b))
        d = np.float32(a + np.float32(c))
    if not np.isfinite(a):
        return None
    if np.isinf(d):              # u/2^24 < a/inf = 0 never holds
        return False
    # u/2^24 < a/d  <=>  u*d < a*2^24   (d > 0)
    return Fraction(int(u)) * Fraction(float(d)) < Fraction(float(a)) * (1 << 24)


def check_decide_exact(libs: Libs):
    gold = json.load(open(os.path.join(GOLDEN, "eq9_threshold_cases.json")))
    for case in gold["cases"]:
        got = oracle.decide(case["u"], case["v"], case["c"], case["eps_b"], lib=libs.f32)
        assert got == case["send"], case
    rng = np.random.default_rng(9)
    for _ in range(4000):
        v = float(np.float32(10 ** rng.uniform(-4, 3)))
        c = float(np.float32(10 ** rng.uniform(-4, 3))) if rng.random() < 0.9 else 0.0
        eps_b = float(np.float32(rng.choice([0.0, 1e-8, 1e-3])))
        a = float(np.float32(np.float32(v) + np.float32(eps_b)))
        d = float(np.float32(np.float32(a) + np.float32(c)))
        if rng.random() < 0.5:      # aim at the threshold: ties and near-ties
            u = int(np.clip(round(a * 2 ** 24 / d) + int(rng.integers(-2, 3)), 0, 2 ** 24 - 1))
        else:
            u = int(rng.integers(0, 2 ** 24))
        want = _exact_decide(u, v, c, eps_b)
        got = oracle.decide(u, v, c, eps_b, lib=libs.f32)
        assert got == want, (u, v, c, eps_b)
    # The whole fp32 range: a and c from subnormal to near FLT_MAX, c = 0 and
    # c = +inf, draws aimed at the threshold.
    for _ in range(4000):
        v = float(np.float32(2.0 ** rng.uniform(-149, 127.9)))
        r = rng.random()
        c = 0.0 if r < 0.1 else float("inf") if r < 0.15 else float(np.float32(2.0 ** rng.uniform(-149, 127.9)))
        eps_b = float(np.float32(rng.choice([0.0, 1e-8, 2.0 ** -140])))
        with np.errstate(over="ignore"):
            a = float(np.float32(np.float32(v) + np.float32(eps_b)))
            d = float(np.float32(np.float32(a) + np.float32(c)))
        if np.isfinite(d) and d > 0 and rng.random() < 0.7:
            u = int(np.clip(int(Fraction(a) * (1 << 24) / Fraction(d)) + int(rng.integers(-2, 3)), 0, 2 ** 24 - 1))
        else:
            u = int(rng.integers(0, 2 ** 24))
        want = _exact_decide(u, v, c, eps_b)
        got = oracle.decide(u, v, c, eps_b, lib=libs.f32)
        assert got == want, (u, v, c, eps_b)
    # Threshold ties constructed exactly: a = 2^k, d = 2^m.
    for k in range(-3, 4):
        for m in range(k, k + 6):
            a, d = 2.0 ** k, 2.0 ** m
            u_tie = int(2 ** 24 * a / d)
            if u_tie >= 2 ** 24 or u_tie < 1:
                continue
            c = d - a
            assert oracle.decide(u_tie, a, c, 0.0, lib=libs.f32) is False
            assert oracle.decide(u_tie - 1, a, c, 0.0, lib=libs.f32) is True


# --------------------------------------------------------------------------
# Philox4x32-10 known-answer vectors and the draw layout
# --------------------------------------------------------------------------
def check_philox_kat(libs: Libs):
    gold = json.load(open(os.path.join(GOLDEN, "philox4x32_10_kat.json")))
    for vec in gold["vectors"]:
        ctr = [int(x, 16) for x in vec["ctr"]]
        key = [int(x, 16) for x in vec["key"]]
        want = [int(x, 16) for x in vec["out"]]
        assert oracle.philox4x32_10(ctr, key, lib=libs.f32) == want, vec


def check_draw_layout_and_uniformity(libs: Libs):
    seed = 0x1234_5678_9ABC_DEF0
    client, push_no = 7, (3 << 32) + 5
    for p in (0, 1, 2, 3, 4, 5, 1023, 4 * 12345 + 2):
        block = oracle.philox4x32_10([p >> 2, client, push_no & 0xFFFFFFFF, push_no >> 32],
                                     [seed & 0xFFFFFFFF, seed >> 32], lib=libs.f32)
        assert oracle.draw(seed, client, push_no, p, lib=libs.f32) == block[p & 3] >> 8
    # Uniformity of u over [0, 2^24): chi-square on 64 bins, 64k draws.
    us = np.array([oracle.draw(seed, 1, 2, p, lib=libs.f32) for p in range(1 << 16)])
    assert us.max() < (1 << 24) and us.min() >= 0
    hist = np.bincount(us >> 18, minlength=64)
    exp = us.size / 64
    chi2 = float(((hist - exp) ** 2 / exp).sum())
    assert chi2 < 130, chi2          # 63 dof: p ~ 1e-6 above 130
    # Different clients / push numbers give unrelated draws.
    a = np.array([oracle.draw(seed, 1, 2, p, lib=libs.f32) for p in range(4096)])
    b = np.array([oracle.draw(seed, 2, 2, p, lib=libs.f32) for p in range(4096)])
    c = np.array([oracle.draw(seed, 1, 3, p, lib=libs.f32) for p in range(4096)])
    assert abs(np.corrcoef(a, b)[0, 1]) < 0.08 and abs(np.corrcoef(a, c)[0, 1]) < 0.08


# --------------------------------------------------------------------------
# B-FASGD select / compact
# --------------------------------------------------------------------------
def check_select_properties(libs: Libs):
    rng = np.random.default_rng(21)
    P = 20001
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)
    v = (10 ** rng.uniform(-1, 2, P)).astype(np.float32)
    seed, eps_b = 77, 1e-8
    # c = 0 keeps everything, in order, bit-copied.
    idx, val = oracle.select(g, v, 0.0, eps_b, seed, 3, 0, lib=libs.f32)
    assert np.array_equal(idx, np.arange(P, dtype=np.int32))
    assert np.array_equal(val.view(np.uint32), g.view(np.uint32))
    # A huge or infinite c keeps nothing.
    for c in (3e38, float("inf")):
        idx, _ = oracle.select(g, v, c, eps_b, seed, 3, 0, lib=libs.f32)
        assert idx.size == 0
    # Moderate c: ascending unique indices, bit-copied values, and a count
    # within 5 sigma of the expected sum of the per-parameter probabilities.
    for c in (1.0, 10.0, 60.0):
        idx, val = oracle.select(g, v, c, eps_b, seed, 5, 9, lib=libs.f32)
        assert np.all(np.diff(idx.astype(np.int64)) > 0)
        assert np.array_equal(val.view(np.uint32), g[idx].view(np.uint32))
        a = v.astype(np.float64) + eps_b
        t = 1.0 / (1.0 + c / a)
        mu, sd = t.sum(), math.sqrt((t * (1 - t)).sum())
        assert abs(idx.size - mu) <= 5 * sd, (c, idx.size, mu, sd)
        # Every index kept satisfies Eq. 9 for its own draw, and every index
        # dropped violates it (checked with exact rationals on a sample).
        keep = np.zeros(P, bool)
        keep[idx] = True
        for p in rng.choice(P, 300, replace=False):
            u = oracle.draw(seed, 5, 9, int(p), lib=libs.f32)
            assert _exact_decide(u, v[p], c, eps_b) == keep[p]


def check_bfasgd_c0_equals_fasgd(libs: Libs):
    rng = np.random.default_rng(8)
    P = 301
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    dense = _server(libs, "f32", P, FASGD)
    sparse = _server(libs, "f32", P, FASGD, c_push=0.0)
    for s in (dense, sparse):
        s.set_params(theta0)
    for t in range(20):
        g = (rng.standard_normal(P) * 0.05).astype(np.float32)
        j = dense.T - min(t % 3, dense.T)
        dense.push(t % 4, j, g)
        idx, val = sparse.select_compact(t % 4, g)
        sparse.push_sparse(t % 4, j, idx, val)
        dense.apply_pending(1)
        sparse.apply_pending(1)
    for x, y in zip(dense.state()[:4], sparse.state()[:4]):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))


def check_sparse_leaves_unsent_untouched(libs: Libs):
    rng = np.random.default_rng(13)
    P = 50
    s = _server(libs, "f32", P, FASGD)
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    s.set_params(theta0)
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)
    s.push(0, 0, g)
    s.apply_pending(1)
    before = [x.copy() for x in s.state()[:4]]
    idx = np.array([1, 5, 6, 40], dtype=np.int32)
    s.push_sparse(0, 1, idx, g[idx])
    s.apply_pending(1)
    after = s.state()[:4]
    mask = np.ones(P, bool)
    mask[idx] = False
    for x, y in zip(before, after):
        assert np.array_equal(x[mask], y[mask])
        assert not np.array_equal(x[idx], y[idx])


def check_fetch_path(libs: Libs):
    """B-FASGD per-parameter fetch: Eq. 9 with the fetch threshold on its own
    draw stream; the client overwrites only the fetched parameters."""
    rng = np.random.default_rng(31)
    P = 12001
    theta = (rng.standard_normal(P) * 0.01).astype(np.float32)
    v = (10 ** rng.uniform(-1, 2, P)).astype(np.float32)
    seed, eps_b = 4242, 1e-8
    # c = 0 fetches everything: the client ends up with the server's theta.
    idx, val = oracle.fetch_select(theta, v, 0.0, eps_b, seed, 2, 0, lib=libs.f32)
    assert np.array_equal(idx, np.arange(P, dtype=np.int32))
    client = np.zeros(P, np.float32)
    oracle.fetch_apply(client, idx, val, lib=libs.f32)
    assert np.array_equal(client.view(np.uint32), theta.view(np.uint32))
    # c = inf fetches nothing.
    idx, _ = oracle.fetch_select(theta, v, float("inf"), eps_b, seed, 2, 0, lib=libs.f32)
    assert idx.size == 0
    # Moderate c: exact Eq. 9 membership on the fetch stream, binomial count,
    # unfetched client entries untouched.
    for c in (5.0, 40.0):
        idx, val = oracle.fetch_select(theta, v, c, eps_b, seed, 3, 7, lib=libs.f32)
        assert np.all(np.diff(idx.astype(np.int64)) > 0)
        assert np.array_equal(val.view(np.uint32), theta[idx].view(np.uint32))
        a = v.astype(np.float64) + eps_b
        t = 1.0 / (1.0 + c / a)
        assert abs(idx.size - t.sum()) <= 5 * math.sqrt((t * (1 - t)).sum())
        keep = np.zeros(P, bool)
        keep[idx] = True
        for p in rng.choice(P, 300, replace=False):
            u = oracle.draw_stream(seed, 1, 3, 7, int(p), lib=libs.f32)
            assert _exact_decide(u, v[p], c, eps_b) == keep[p]
        stale = np.full(P, 7.0, np.float32)
        oracle.fetch_apply(stale, idx, val, lib=libs.f32)
        assert np.all(stale[~keep] == 7.0) and np.array_equal(stale[keep], theta[keep])
    # The fetch stream is not the push stream.
    same = [oracle.draw_stream(seed, 0, 3, 7, p, lib=libs.f32) ==
            oracle.draw_stream(seed, 1, 3, 7, p, lib=libs.f32) for p in range(2000)]
    assert sum(same) < 5
    assert oracle.draw_stream(seed, 0, 3, 7, 11, lib=libs.f32) == oracle.draw(seed, 3, 7, 11,
                                                                              lib=libs.f32)


def check_server_fetch_counters(libs: Libs):
    s = _server(libs, "f32", 64, FASGD, lam=3)
    s.set_fetch_threshold(1.0)
    g = np.ones(64, np.float32)
    s.select_compact(1, g)
    s.fetch_compact(1)
    s.fetch_compact(1)
    assert s.push_count == [0, 1, 0] and s.fetch_count == [0, 2, 0]
    a = s.fetch_compact(2)
    b = oracle.fetch_select(s.theta, s.v, 1.0, s.eps_b, s.seed, 2, 0, lib=libs.f32)
    assert np.array_equal(a[0], b[0])


# --------------------------------------------------------------------------
# Exact means (the per-message and per-tensor statistics)
# --------------------------------------------------------------------------
def _exact_sum(x) -> Fraction:
    """The exact sum of fp32 (or fp64) values: each is m 2^e with an integer
    significand m, so grouping by exponent sums integers only."""
    x = np.asarray(x, dtype=np.float64)
    assert np.isfinite(x).all()
    m, e = np.frexp(x)                       # x = m 2^e, 1/2 <= |m| < 1
    mi = (m * 2.0 ** 53).astype(np.int64)    # exact: a double has 53 significant bits
    total = 0
    for ee in np.unique(e):                  # x = mi 2^(e - 53); units of 2^-1127
        total += int(mi[e == ee].astype(object).sum()) << int(ee - 53 + 1127)
    return Fraction(total, 1 << 1127)


def _f32_nearest(q: Fraction) -> np.float32:
    """The fp32 value nearest to the rational q, ties to the even
    significand: q is compared exactly with a first guess and its two
    neighbours (the guess, q rounded through fp64, is within one step)."""
    guess = np.float32(float(q))
    best = None
    for x in (np.nextafter(guess, np.float32(-np.inf)), guess,
              np.nextafter(guess, np.float32(np.inf))):
        if not np.isfinite(x):
            continue
        key = (abs(Fraction(float(x)) - q), int(x.view(np.uint32)) & 1)
        if best is None or key < best[0]:
            best = (key, x)
    return best[1]


def _check_exact_means(libs: Libs, mean):
    """mean(v, real) -> fp32: the exact mean of v rounded once, for more than
    a million terms and at constructed rounding boundaries."""
    rng = np.random.default_rng(47)
    P = 1_000_003
    v = (10 ** rng.uniform(-3, 3, P)).astype(np.float32)
    v[rng.random(P) < 0.01] = 0.0
    want = _f32_nearest(_exact_sum(v) / P)
    for real in ("f32", "f64"):
        assert mean(v, real) == want, real
    # Values on an fp32 rounding boundary: (P - 2) copies of lo, z1 and z2
    # with an exact sum of P (lo + up) / 2 + delta, up the float after lo.
    # delta = 0 is a tie (to the even one of lo and up); delta = +-2^-149 puts
    # the mean just above or below it, by far less than an fp64 sum of a
    # million terms near 1.5 can resolve.
    # With P = 2^20 the excess delta / P is a whole number of units of the
    # exact quotient (no remainder); with P = 3 2^19 it is not.
    tiny = np.float32(2.0 ** -149)
    for P in (3 << 19, 1 << 20):
        for lo in (np.float32(1.5), np.nextafter(np.float32(1.5), np.float32(2))):
            up = np.nextafter(lo, np.float32(2))
            gap = P * (Fraction(float(up)) - Fraction(float(lo))) / 2
            z1 = np.float32(2 * Fraction(float(lo)) + gap)
            assert Fraction(float(z1)) == 2 * Fraction(float(lo)) + gap
            even = lo if int(lo.view(np.uint32)) % 2 == 0 else up
            for delta, expect in ((np.float32(0.0), even), (tiny, up), (-tiny, lo)):
                v = np.full(P, lo, dtype=np.float32)
                v[P // 3] = z1
                v[-1] = delta
                assert _f32_nearest(_exact_sum(v) / P) == expect
                for real in ("f32", "f64"):
                    assert mean(v, real) == expect, (real, P, float(lo), float(delta))
    P = 3 << 19
    # In the fp64 build the terms are doubles: a term of 2^-1074 moves the
    # mean by less than one unit of the exact quotient, so only the remainder
    # of the division can tell that it is above the tie.
    lo = np.float32(1.5)
    up = np.nextafter(lo, np.float32(2))
    v = np.full(P, float(lo))
    v[P // 3] = float(np.float32(2 * Fraction(float(lo)) + P * (Fraction(float(up)) - Fraction(float(lo))) / 2))
    v[-1] = 2.0 ** -1074
    assert mean(v, "f64") == up
    # Signs, zeros and subnormals: the exact mean of a mixed vector.
    v = (rng.standard_normal(4099) * 10.0 ** rng.integers(-45, 3, 4099)).astype(np.float32)
    for real in ("f32", "f64"):
        assert mean(v, real) == _f32_nearest(_exact_sum(v) / v.size), real
        assert mean(np.zeros(5, np.float32), real) == 0.0


def check_message_path(libs: Libs):
    """The paper's literal B-FASGD (Sec. 2.3): one Eq. 9 decision per message
    against the mean of v; dropped pushes re-apply the client's cached
    gradient; dropped fetches leave the client's copy as it is."""
    rng = np.random.default_rng(41)
    # The statistic is the exact mean of v, rounded once to fp32.
    for real in ("f32", "f64"):
        for P in (1, 7, 1000, 4099):
            v = (10 ** rng.uniform(-2, 3, P)).astype(np.float32)
            got = oracle.mean_v(v, real, lib=libs.lib(real))
            assert np.float32(got) == _f32_nearest(_exact_sum(v) / P), (real, P)
    _check_exact_means(libs, lambda v, real: np.float32(oracle.mean_v(v, real, lib=libs.lib(real))))
    # Message draws are their own domain (not the per-parameter draws).
    seed = 99
    same = sum(oracle.draw_message(seed, 0, 2, n, lib=libs.f32) ==
               oracle.draw_stream(seed, 0, 2, n, 0, lib=libs.f32) for n in range(300))
    assert same < 3
    assert sum(oracle.draw_message(seed, 0, 2, n, lib=libs.f32) ==
               oracle.draw_message(seed, 1, 2, n, lib=libs.f32) for n in range(300)) < 3
    P, lam = 37, 3
    grads = [(rng.standard_normal(P) * 0.1).astype(np.float32) for _ in range(30)]
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)

    def run(c_push, variant=FASGD):
        s = _server(libs, "f32", P, variant, lam=lam, c_push=c_push, seed=seed)
        s.set_params(theta0)
        for t, g in enumerate(grads):
            s.push_message(t % lam, s.T - min(t % 2, s.T), g)
            s.apply_pending(1)
        return s

    def dense(seq, variant=FASGD):
        s = _server(libs, "f32", P, variant, lam=lam)
        s.set_params(theta0)
        for t, g in enumerate(seq):
            s.push(t % lam, s.T - min(t % 2, s.T), g)
            s.apply_pending(1)
        return s

    # c = 0: every push is sent -> plain FASGD.
    a, b = run(0.0), dense(grads)
    assert all(a.message_log)
    for x, y in zip(a.state()[:4], b.state()[:4]):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    # c = inf: nothing is sent, nothing is cached -> zero gradients.
    a, b = run(float("inf")), dense([np.zeros(P, np.float32)] * len(grads))
    assert not any(a.message_log)
    for x, y in zip(a.state()[:4], b.state()[:4]):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    # Moderate c: the run equals plain FASGD on the sequence where each dropped
    # push is replaced by its client's last sent gradient.
    a = run(30.0)
    assert 0 < sum(a.message_log) < len(grads)
    last, seq = {}, []
    for t, (g, sent) in enumerate(zip(grads, a.message_log)):
        c = t % lam
        if sent:
            last[c] = g
        seq.append(last.get(c, np.zeros(P, np.float32)))
    b = dense(seq)
    for x, y in zip(a.state()[:4], b.state()[:4]):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    # Decisions are Eq. 9 against the mean of v, with the message draw; the
    # send fraction at fixed v matches 1 / (1 + c / v).
    s = _server(libs, "f32", P, ASGD, lam=1, c_push=4.0, seed=seed)
    s.v[:] = 4.0                     # ASGD never changes v
    for t in range(3000):
        s.push_message(0, s.T, grads[t % len(grads)])
        s.apply_pending(1)
    for n in range(50):
        u = oracle.draw_message(seed, 0, 0, n, lib=libs.f32)
        assert s.message_log[n] == _exact_decide(u, 4.0, 4.0, s.eps_b)
    frac = sum(s.message_log) / 3000
    assert abs(frac - 0.5) < 5 * math.sqrt(0.25 / 3000), frac
    # Fetch messages: c_fetch = 0 always fetches, inf never.
    s = _server(libs, "f32", P, FASGD, lam=2, seed=seed)
    s.push(0, 0, grads[0])
    s.apply_pending(1)
    copy = np.full(P, 3.0, np.float32)
    s.set_fetch_threshold(float("inf"))
    assert s.fetch_message(1, copy) is False and np.all(copy == 3.0)
    s.set_fetch_threshold(0.0)
    assert s.fetch_message(1, copy) is True
    assert np.array_equal(copy.view(np.uint32), s.theta.view(np.uint32))
    assert s.fetch_count == [0, 2]


def check_sim_objective(libs: Libs):
    """The closed-loop simulation's objective: the deterministic part of the
    gradient is h (theta - star) in fp32, the noise is uniform with the stated
    variance and range, fresh per (client, gradient count), and the loss is
    1/2 sum h (theta - star)^2; a single client with full fetches reproduces
    plain stochastic gradient descent step by step."""
    import oracle.sim as osim
    rng = np.random.default_rng(51)
    P = 50_000
    th = (rng.standard_normal(P) * 0.1).astype(np.float32)
    h = (10 ** rng.uniform(-2, 1, P)).astype(np.float32)
    star = (rng.standard_normal(P) * 0.1).astype(np.float32)
    g = oracle.sim_grad(th, h, star, np.zeros(P, np.float32), 5, 1, 0, lib=libs.f32)
    assert np.array_equal(g.view(np.uint32), (h * (th - star)).astype(np.float32).view(np.uint32))
    sig = np.full(P, 0.25, np.float32)
    noise = oracle.sim_grad(star, h, star, sig, 5, 1, 0, lib=libs.f32).astype(np.float64)
    assert abs(noise.mean()) < 5 * 0.25 / math.sqrt(P)
    assert abs(noise.var() - 0.0625) < 0.0625 * 0.03
    assert np.max(np.abs(noise)) <= 0.25 * math.sqrt(3) * (1 + 1e-6)
    other = oracle.sim_grad(star, h, star, sig, 5, 2, 0, lib=libs.f32)
    again = oracle.sim_grad(star, h, star, sig, 5, 1, 0, lib=libs.f32)
    later = oracle.sim_grad(star, h, star, sig, 5, 1, 1, lib=libs.f32)
    assert np.array_equal(again, noise.astype(np.float32))
    assert abs(np.corrcoef(noise, other)[0, 1]) < 0.02 and abs(np.corrcoef(noise, later)[0, 1]) < 0.02
    terms = (h * ((th - star) * (th - star))).astype(np.float32).astype(np.float64)
    want = 0.5 * math.fsum(terms)
    assert abs(oracle.sim_loss(th, h, star, lib=libs.f32) - want) <= 1e-12 * want
    # One client, full fetches: the simulation is plain SGD at the current point.
    Ps = 301
    obj = (h[:Ps], star[:Ps], (10 ** rng.uniform(-3, -1, Ps)).astype(np.float32))
    th0 = np.zeros(Ps, np.float32)
    sim = osim.OracleSimulation(Ps, 1, 0.05, ASGD, objective=obj, theta0=th0, seed=3,
                                lib=libs.f32)
    sim.run(np.zeros((40, 1), np.int32))
    ref = th0.copy()
    a32 = np.float32(0.05)
    for t in range(40):
        gt = oracle.sim_grad(ref, *obj, 3, 0, t, lib=libs.f32)
        ref = (ref - a32 * gt).astype(np.float32)
    assert np.array_equal(sim.srv.theta.view(np.uint32), ref.view(np.uint32))


def check_sim_protocol(libs: Libs):
    """The closed-loop simulation with several clients, restated plainly:
    every client keeps a copy of the parameters and the server timestamp it
    was taken at; a dispatcher batch of clients computes gradients at their
    copies (noise drawn per client and gradient count), pushes them with
    those timestamps, the server applies the batch in order (push k at
    T + k: tau = T + k - j), and the clients of the batch then refresh.  A
    full refresh, and the per-parameter, per-message and per-tensor refreshes
    at the thresholds or budgets that fetch everything or nothing, reproduce
    the restatement bit for bit under ASGD and SASGD.  (A per-parameter or
    per-tensor refresh stamps the copy with T whatever it transmitted; a
    per-message refresh only when it fetches.)"""
    import oracle.sim as osim
    rng = np.random.default_rng(97)
    P, lam, seed = 37, 3, 11
    obj = ((10 ** rng.uniform(-1, 0.5, P)).astype(np.float32),
           (rng.standard_normal(P) * 0.1).astype(np.float32),
           (10 ** rng.uniform(-3, -1, P)).astype(np.float32))
    th0 = (rng.standard_normal(P) * 0.1).astype(np.float32)
    schedule = [[0], [1], [0, 2], [1, 2, 0], [2], [0, 1], [1], [2, 0]]
    a32 = np.float32(0.05)

    def restated(variant, copy_refresh, stamp_refresh):
        theta, T = th0.copy(), 0
        copies = [th0.copy() for _ in range(lam)]
        stamp, count = [0] * lam, [0] * lam
        for batch in schedule:
            pushes = []
            for c in batch:
                pushes.append((stamp[c], oracle.sim_grad(copies[c], *obj, seed, c, count[c],
                                                         lib=libs.f32)))
                count[c] += 1
            for k, (j, g) in enumerate(pushes):
                tau = T + k - j
                coef = a32 if variant == ASGD else np.float32(float(a32) / max(tau, 1))
                theta = (theta - coef * g).astype(np.float32)
            T += len(batch)
            for c in batch:
                if copy_refresh:
                    copies[c] = theta.copy()
                if stamp_refresh:
                    stamp[c] = T
        return theta

    inf = float("inf")
    cases = [("full", {}, True, True),
             ("param", {"c_fetch": 0.0}, True, True), ("param", {"c_fetch": inf}, False, True),
             ("message", {"c_fetch": 0.0}, True, True), ("message", {"c_fetch": inf}, False, False),
             ("budget", {"fetch_budget": P, "tensor_sizes": [10, 27]}, True, True),
             ("budget", {"fetch_budget": 0, "tensor_sizes": [10, 27]}, False, True)]
    for variant in (ASGD, SASGD):
        for fetch, kw, copy_refresh, stamp_refresh in cases:
            sim = osim.OracleSimulation(P, lam, float(a32), variant, objective=obj, theta0=th0,
                                        seed=seed, fetch=fetch, lib=libs.f32, **kw)
            sim.run(schedule)
            want = restated(variant, copy_refresh, stamp_refresh)
            assert np.array_equal(sim.srv.theta.view(np.uint32), want.view(np.uint32)), (
                variant, fetch, kw)
    # the restatement itself sees the staleness: SASGD differs from ASGD here
    assert not np.array_equal(restated(ASGD, True, True), restated(SASGD, True, True))


def check_protocol_errors(libs: Libs):
    s = _server(libs, "f32", 4, FASGD, lam=2)
    g = np.zeros(4, np.float32)
    for bad in ((2, 0), (-1, 0), (0, 1), (0, -1)):
        try:
            s.push(bad[0], bad[1], g)
        except oracle.OracleError:
            pass
        else:
            raise AssertionError(f"push {bad} accepted")
    try:
        s.apply_pending(1)
    except oracle.OracleError:
        pass
    else:
        raise AssertionError("apply with empty queue accepted")
    s.push(0, 0, g)
    try:
        s.push_sparse(0, 0, np.array([2, 1], np.int32), np.zeros(2, np.float32))
        s.apply_pending(2)
    except oracle.OracleError:
        pass
    else:
        raise AssertionError("descending sparse list accepted")
    t = _server(libs, "f32", 4, FASGD, lam=2)
    for bad in (lambda: t.push_budget(0, 0, g, 2),          # no partition yet
                lambda: t.set_tensors([1, 2]),               # sizes do not sum to P
                lambda: t.set_tensors([4, 0]),               # empty tensor
                lambda: (t.set_tensors([1, 3]), t.push_budget(0, 0, g, -1))):
        try:
            bad()
        except (oracle.OracleError, AssertionError):
            pass
        else:
            raise AssertionError("bad per-tensor call accepted")


# --------------------------------------------------------------------------
# Per-tensor B-FASGD under a bandwidth budget (future-work section)
# --------------------------------------------------------------------------
def _budget_E(sizes, vbar, eps_b, x):
    """E(x) from its definition, independently: numpy's IEEE fp32 add and
    divide for q_t, then exact rationals for floor(s_t q_t 2^32)."""
    tot = 0
    with np.errstate(over="ignore", invalid="ignore", divide="ignore"):
        for s, vb in zip(sizes, vbar):
            a = np.float32(vb) + np.float32(eps_b)
            if not (a > 0 and np.isfinite(a)):
                continue
            q = a / (a + np.float32(x))
            tot += math.floor(Fraction(float(q)) * int(s) * 2 ** 32)
    return tot


def _f32_prev(x):
    return float(np.array([np.float32(x).view(np.uint32) - 1], np.uint32).view(np.float32)[0])


def _budget_instances(rng, n):
    for k in range(n):
        T = int(rng.integers(1, 13))
        sizes = rng.integers(1, 5000, T)
        sizes[rng.random(T) < 0.2] = 1
        vbar = (10 ** rng.uniform(-3, 3, T)).astype(np.float32)
        eps_b = (0.0, 1e-8, 0.5)[k % 3]
        if eps_b == 0.0:
            vbar[rng.random(T) < 0.2] = 0.0       # a_t = 0: never sent, no share
        S = int(sizes.sum())
        for B in (0, 1, S // 7, S // 2, S - 1, S, S + 10):
            yield sizes, vbar, eps_b, max(B, 0)


def check_tensor_means(libs: Libs):
    """vbar_t is the exact mean of v over tensor t, rounded once to fp32."""
    rng = np.random.default_rng(61)
    for real in ("f32", "f64"):
        sizes = np.array([1, 7, 1000, 4099, 2, 333])
        v = (10 ** rng.uniform(-2, 3, int(sizes.sum()))).astype(np.float32)
        got = oracle.tensor_means(v, sizes, real, lib=libs.lib(real))
        off = np.concatenate([[0], np.cumsum(sizes)])
        for t in range(sizes.size):
            seg = v[off[t]:off[t + 1]]
            assert got[t] == _f32_nearest(_exact_sum(seg) / int(sizes[t])), (real, t)
        assert got[0] == v[0]                          # one-element tensor: v itself
        const = np.repeat(np.float32([0.3, 7.0, 1e-3]), [5, 11, 3])
        assert np.array_equal(oracle.tensor_means(const, [5, 11, 3], real, lib=libs.lib(real)),
                              np.float32([0.3, 7.0, 1e-3]))
    # One tensor over everything: the per-message statistic.
    v = (10 ** rng.uniform(-2, 3, 5000)).astype(np.float32)
    assert oracle.tensor_means(v, [5000], lib=libs.f32)[0] == oracle.mean_v(v, lib=libs.f32)

    # The same constructions as the per-message statistic, each as the middle
    # tensor of three (so the offsets matter too).
    def middle(v, real):
        sizes = [3, v.shape[0], 5]
        w = np.concatenate([np.full(3, 7.0), np.asarray(v, dtype=np.float64), np.full(5, 1e-3)])
        return oracle.tensor_means(w, sizes, real, lib=libs.lib(real))[1]
    _check_exact_means(libs, middle)


def check_budget_threshold(libs: Libs):
    """c is the smallest non-negative float (or +inf) with E(c) <= B 2^32,
    E defined exactly; equal statistics give the closed form a (S/B - 1)."""
    rng = np.random.default_rng(62)
    for sizes, vbar, eps_b, B in _budget_instances(rng, 24):
        S = int(sizes.sum())
        limit = min(B, S) * 2 ** 32
        c = oracle.budget_c(sizes, vbar, eps_b, B, lib=libs.f32)
        assert c >= 0.0
        e_c = _budget_E(sizes, vbar, eps_b, c)
        assert oracle.budget_expected(sizes, vbar, eps_b, c, lib=libs.f32) == e_c
        assert e_c <= limit, (B, c)
        if c > 0.0:
            prev = _f32_prev(c)
            e_prev = _budget_E(sizes, vbar, eps_b, prev)
            assert oracle.budget_expected(sizes, vbar, eps_b, prev, lib=libs.f32) == e_prev
            assert e_prev > limit, (B, c, prev)
        for x in (0.0, 1e-3, 1.0, 123.5, 3e38, float("inf")):
            assert oracle.budget_expected(sizes, vbar, eps_b, x, lib=libs.f32) == \
                _budget_E(sizes, vbar, eps_b, x)
        if B >= S and (vbar.astype(np.float64) + eps_b > 0).all():
            assert c == 0.0
    # Non-increasing in the budget.
    sizes = np.array([100, 2000, 5, 40000])
    vbar = np.float32([0.5, 3.0, 40.0, 0.01])
    cs = [oracle.budget_c(sizes, vbar, 0.0, B, lib=libs.f32) for B in range(0, 42106, 1000)]
    assert all(x >= y for x, y in zip(cs, cs[1:]))
    # Equal statistics: sum_t s_t a / (a + c) = B  =>  c = a (S / B - 1).
    for a, B in ((0.7, 2500), (13.0, 9000), (2e-3, 100)):
        sizes = np.array([1000, 3000, 6000])
        c = oracle.budget_c(sizes, np.float32([a] * 3), 0.0, B, lib=libs.f32)
        want = float(np.float32(a)) * (10000 / B - 1)
        assert abs(c - want) <= 2e-6 * want, (a, B, c, want)


def check_tensor_decisions(libs: Libs):
    """Tensor draws have their own Philox domain and layout; decisions are
    Eq. 9 per tensor; over many pushes the parameters sent average E(c)."""
    seed, client = 0xFEED_F00D_1234, 5
    for stream in (0, 1):
        for n in (0, 1, (2 << 32) + 9):
            for t in (0, 1, 2, 3, 4, 4099):
                block = oracle.philox4x32_10(
                    [(1 << 31) + (t >> 2), client | (stream << 31), n & 0xFFFFFFFF, n >> 32],
                    [seed & 0xFFFFFFFF, seed >> 32], lib=libs.f32)
                assert oracle.draw_tensor(seed, stream, client, n, t, lib=libs.f32) == \
                    block[t & 3] >> 8
    same = sum(oracle.draw_tensor(seed, 0, 2, n, 0, lib=libs.f32) ==
               oracle.draw_stream(seed, 0, 2, n, 0, lib=libs.f32) for n in range(300))
    assert same < 3
    sizes = np.array([10, 700, 3000, 1, 64, 20000, 5, 900])
    vbar = np.float32([0.1, 4.0, 1.0, 50.0, 0.5, 2.0, 0.02, 9.0])
    eps_b = 1e-8
    S = int(sizes.sum())
    B = S // 4
    c = oracle.budget_c(sizes, vbar, eps_b, B, lib=libs.f32)
    N = 3000
    tot = []
    for n in range(N):
        sent, m = oracle.tensor_select(sizes, vbar, c, eps_b, seed, 0, client, n, lib=libs.f32)
        assert m == int((sizes * sent).sum())
        if n < 40:
            for t in range(sizes.size):
                u = oracle.draw_tensor(seed, 0, client, n, t, lib=libs.f32)
                assert bool(sent[t]) == _exact_decide(u, vbar[t], c, eps_b)
        tot.append(m)
    q = np.array([float(np.float32(vb + np.float32(eps_b)) / np.float32(np.float32(vb + np.float32(eps_b)) + np.float32(c)))
                  for vb in vbar])
    mu = float((sizes * q).sum())
    sd = math.sqrt(float((sizes.astype(np.float64) ** 2 * q * (1 - q)).sum()) / N)
    assert abs(np.mean(tot) - mu) <= 5 * sd + S * 2.0 ** -24, (np.mean(tot), mu, sd)
    assert abs(mu - B) <= 1.0
    # c = 0 sends every tensor; c = +inf none.
    assert oracle.tensor_select(sizes, vbar, 0.0, eps_b, seed, 0, 1, 0, lib=libs.f32)[1] == S
    assert oracle.tensor_select(sizes, vbar, float("inf"), eps_b, seed, 0, 1, 0,
                                lib=libs.f32)[1] == 0


def check_budget_server(libs: Libs):
    """Server path: a budget of P or more is plain FASGD; a zero budget
    changes nothing but T; otherwise the run equals sparse pushes of exactly
    the transmitted tensors, each decided against the v of that moment."""
    rng = np.random.default_rng(63)
    sizes = np.array([40, 3, 17, 1, 60, 9])
    P, lam, seed = int(sizes.sum()), 3, 2024
    off = np.concatenate([[0], np.cumsum(sizes)])
    grads = [(rng.standard_normal(P) * 0.1).astype(np.float32) for _ in range(25)]
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)

    def run(budget, variant=FASGD):
        s = _server(libs, "f32", P, variant, lam=lam, seed=seed, eps_b=1e-3)
        s.set_params(theta0)
        s.set_tensors(sizes)
        for t, g in enumerate(grads):
            s.push_budget(t % lam, s.T - min(t % 2, s.T), g, budget)
            s.apply_pending(1)
        return s

    for variant in (FASGD, FASGD_STD, SASGD):
        a = run(P + 5, variant)
        assert all(log[0].all() and log[1] == 0.0 and log[2] == P for log in a.budget_log)
        b = _server(libs, "f32", P, variant, lam=lam)
        b.set_params(theta0)
        for t, g in enumerate(grads):
            b.push(t % lam, b.T - min(t % 2, b.T), g)
            b.apply_pending(1)
        for x, y in zip(a.state(), b.state()):
            assert np.array_equal(np.asarray(x).view(np.uint32) if hasattr(x, "view") else x,
                                  np.asarray(y).view(np.uint32) if hasattr(y, "view") else y)
    a = run(0)
    assert a.T == len(grads) and sum(int(log[0].sum()) for log in a.budget_log) == 0
    assert np.array_equal(a.theta, theta0) and not a.v.any() and not a.n.any()
    # Moderate budget, replayed as sparse pushes of the transmitted ranges.
    a = run(P // 3)
    ref = _server(libs, "f32", P, FASGD, lam=lam, seed=seed, eps_b=1e-3)
    ref.set_params(theta0)
    total = 0
    for t, (g, (sent, c, m)) in enumerate(zip(grads, a.budget_log)):
        vbar = oracle.tensor_means(ref.v, sizes, lib=libs.f32)
        assert c == oracle.budget_c(sizes, vbar, 1e-3, P // 3, lib=libs.f32)
        idx = np.concatenate([np.arange(off[k], off[k + 1]) for k in np.flatnonzero(sent)]
                             + [np.zeros(0, np.int64)]).astype(np.int32)
        assert m == idx.size
        total += m
        ref.push_sparse(t % lam, ref.T - min(t % 2, ref.T), idx, g[idx])
        ref.apply_pending(1)
    assert 0 < total < P * len(grads)
    for x, y in zip(a.state()[:4], ref.state()[:4]):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
    assert a.push_count == [9, 8, 8]
    # Fetches: a full budget copies theta, a zero budget copies nothing, and
    # a partial one copies exactly the transmitted tensors.
    copy = np.full(P, 5.0, np.float32)
    assert a.fetch_budget(1, copy, 0)[2] == 0 and np.all(copy == 5.0)
    sent, c, m = a.fetch_budget(1, copy, P // 2)
    for k in range(sizes.size):
        seg = copy[off[k]:off[k + 1]]
        if sent[k]:
            assert np.array_equal(seg, a.theta[off[k]:off[k + 1]])
        else:
            assert np.all(seg == 5.0)
    assert m == int((sizes * sent).sum())
    assert a.fetch_budget(1, copy, P)[2] == P and np.array_equal(copy, a.theta)
    assert a.fetch_count == [0, 3, 0]


# --------------------------------------------------------------------------
# Protocol: batches in arrival order, draws keyed by the right stream and count
# --------------------------------------------------------------------------
def check_batched_apply_order(libs: Libs):
    """Sec. 2.1: queued pushes are applied in arrival order, push k of a batch
    at server timestamp T + k.  Batches of 1 to 5 pushes with mixed staleness
    equal the fp64 series form with tau_k = T + k - j_k; the same pushes in
    reverse arrival order do not."""
    rng = np.random.default_rng(71)
    P = 5
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    gamma, beta, eps, alpha = 0.8, 0.6, 1e-3, 0.05
    sizes = [3, 1, 4, 2, 5]
    batches, T = [], 0
    for k in sizes:
        batch = []
        for _ in range(k):
            g = (rng.standard_normal(P) * rng.choice([0.01, 0.5, 2.0])).astype(np.float32)
            batch.append((T - min(int(rng.integers(0, 4)), T), g))
        batches.append(batch)
        T += k

    def events(order):
        out, T = [], 0
        for batch in batches:
            for k, (j, g) in enumerate(order(batch)):
                out.append((T + k - j, {p: float(g[p]) for p in range(P)}))
            T += len(batch)
        return out

    for variant in (SASGD, FASGD):
        G, B = float(np.float32(gamma)), float(np.float32(beta))
        E, A = float(np.float32(eps)), float(np.float32(alpha))
        ref = _series_reference(variant, theta0, events(lambda b: b), A, G, B, E)
        rev = _series_reference(variant, theta0, events(lambda b: b[::-1]), A, G, B, E)
        assert _rel(rev[0], ref[0]) > 1e-6          # the order is visible in theta
        s = _server(libs, "f64", P, variant, alpha=alpha, gamma=gamma, beta=beta, eps=eps)
        s.set_params(theta0)
        for batch in batches:
            for c, (j, g) in enumerate(batch):
                s.push(c % s.lam, j, g)
            s.apply_pending(len(batch))
        assert s.T == T and not s.fifo
        for name, got, r in zip(("theta", "n", "b", "v"), s.state()[:4], ref):
            bound = 1e-12 * (np.abs(r) + np.max(np.abs(r)) + 1e-30)
            assert np.all(np.abs(got - r) <= bound), (variant, name)


def check_fetch_draws_keyed_by_fetch_count(libs: Libs):
    """A client's n-th per-parameter fetch is decided with the draws of its
    n-th fetch (stream 1), whatever pushes it selected in between: two
    servers in the same state, one of which selects three pushes between its
    fetches, return the same fetch lists; and fetch and push lists of the
    same count differ (separate streams)."""
    rng = np.random.default_rng(83)
    P = 4096
    theta0 = (rng.standard_normal(P) * 0.01).astype(np.float32)
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)

    def server():
        s = _server(libs, "f32", P, FASGD, lam=3, c_push=1.0, seed=555)
        s.set_params(theta0)
        s.push(0, 0, g)
        s.apply_pending(1)
        s.set_fetch_threshold(1.0)
        return s

    a, b = server(), server()
    fa = [a.fetch_compact(2) for _ in range(2)]
    pushes = [b.select_compact(2, g) for _ in range(3)]
    fb = [b.fetch_compact(2)]
    b.select_compact(2, g)
    fb.append(b.fetch_compact(2))
    for (ia, va), (ib, vb) in zip(fa, fb):
        assert np.array_equal(ia, ib) and np.array_equal(va, vb)
    assert 0 < fa[0][0].size < P
    assert not np.array_equal(fa[0][0], pushes[0][0])


def check_tensor_streams_separate(libs: Libs):
    """Per-tensor rule: a client's n-th budget fetch and its n-th budget push,
    decided against the same statistics and budget, draw from separate
    streams -- over 64 tensors their decisions differ."""
    rng = np.random.default_rng(89)
    sizes = rng.integers(1, 40, 64)
    P = int(sizes.sum())
    g = (rng.standard_normal(P) * 0.1).astype(np.float32)

    def server():
        s = _server(libs, "f32", P, FASGD, lam=2, seed=777, eps_b=1e-3)
        s.set_tensors(sizes)
        s.push(0, 0, g)
        s.apply_pending(1)
        return s

    a, b = server(), server()
    copy = np.zeros(P, np.float32)
    sent_fetch, c_fetch, _ = a.fetch_budget(1, copy, P // 2)
    b.push_budget(1, b.T, g, P // 2)
    b.apply_pending(1)
    sent_push, c_push, _ = b.budget_log[-1]
    assert c_fetch == c_push                      # same statistics, same budget
    assert 0 < int(sent_fetch.sum()) < sizes.size
    assert not np.array_equal(sent_fetch, sent_push)


ALL_CHECKS = [  # quick pins first: a mutant stops at the first pin it fails
    check_hand_trace,
    check_constant_gradient_closed_form,
    check_std_variant_closed_form,
    check_series_bruteforce,
    check_variant_invariants,
    check_dense_equals_full_sparse,
    check_decide_exact,
    check_philox_kat,
    check_draw_layout_and_uniformity,
    check_select_properties,
    check_bfasgd_c0_equals_fasgd,
    check_sparse_leaves_unsent_untouched,
    check_fetch_path,
    check_server_fetch_counters,
    check_sim_objective,
    check_budget_threshold,
    check_tensor_decisions,
    check_budget_server,
    check_batched_apply_order,
    check_fetch_draws_keyed_by_fetch_count,
    check_tensor_streams_separate,
    check_sim_protocol,
    check_protocol_errors,
    check_tensor_means,
    check_message_path,
]
