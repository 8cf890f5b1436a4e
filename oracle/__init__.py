"""CPU oracle for the FASGD parameter-server path -- TEST INFRASTRUCTURE ONLY.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may import this package.  The CUDA path never does and
shares no code with it.

``fasgd_oracle.c`` holds the elementwise rules (Eq. 1-2, 4-8, 9 of the
paper); this module compiles it twice (fp32 and fp64 parameter/state type)
and adds the server protocol of Section 2.1 around it as a plain Python
FIFO: a push carries (client, timestamp j, gradient); applying it computes
the step-staleness tau = T - j against the current server timestamp T,
updates every parameter, and increments T.

Parity status: every function here is pinned by the ``-m "not gpu"`` tests
(closed forms, hand traces, series brute force, exact-rational checks of the
send decision, Philox known-answer vectors, invariants between variants).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

ASGD, SASGD, FASGD, FASGD_STD = 0, 1, 2, 3

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fasgd_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LOCK = threading.Lock()
_LIBS: dict = {}

_CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", "-Wall", "-Wextra"]


def lib_path(real: str) -> str:
    return os.path.join(_BUILD, f"libfasgd_oracle_{real}.so")


def build(force: bool = False) -> None:
    """Compile the oracle (fp32 and fp64 builds) with gcc if out of date."""
    os.makedirs(_BUILD, exist_ok=True)
    for real, ctype in (("f32", "float"), ("f64", "double")):
        out = lib_path(real)
        if (not force and os.path.exists(out)
                and os.path.getmtime(out) >= os.path.getmtime(_SRC)):
            continue
        tmp = out + f".tmp{os.getpid()}"
        subprocess.run(["gcc", *_CFLAGS, f"-DREAL={ctype}", _SRC, "-o", tmp, "-lm"],
                       check=True)
        os.replace(tmp, out)


def load_library(path: str, real: str) -> ctypes.CDLL:
    """Load one oracle build and declare its signatures."""
    lib = ctypes.CDLL(path)
    R = ctypes.c_float if real == "f32" else ctypes.c_double
    P = ctypes.c_void_p
    i64, u32, u64, i32 = ctypes.c_int64, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int
    lib.ora_real_bytes.restype = i32
    lib.ora_real_bytes.argtypes = []
    lib.ora_coef.restype = R
    lib.ora_coef.argtypes = [i32, ctypes.c_float, i64]
    lib.ora_apply_dense.restype = None
    lib.ora_apply_dense.argtypes = [i32, i64, P, P, P, P, P, R, R, R, R]
    lib.ora_apply_sparse.restype = i32
    lib.ora_apply_sparse.argtypes = [i32, i64, P, P, P, P, i64, P, P, R, R, R, R]
    lib.ora_philox4x32_10.restype = None
    lib.ora_philox4x32_10.argtypes = [P, P, P]
    lib.ora_draw.restype = u32
    lib.ora_draw.argtypes = [u64, u32, u64, i64]
    lib.ora_decide.restype = i32
    lib.ora_decide.argtypes = [u32, ctypes.c_float, ctypes.c_float, ctypes.c_float]
    lib.ora_select.restype = i64
    lib.ora_select.argtypes = [i64, P, P, ctypes.c_float, ctypes.c_float, u64, u32, u64, P, P]
    lib.ora_draw_stream.restype = u32
    lib.ora_draw_stream.argtypes = [u64, u32, u32, u64, i64]
    lib.ora_fetch_select.restype = i64
    lib.ora_fetch_select.argtypes = [i64, P, P, ctypes.c_float, ctypes.c_float, u64, u32, u64,
                                     P, P]
    lib.ora_fetch_apply.restype = None
    lib.ora_fetch_apply.argtypes = [P, i64, P, P]
    lib.ora_mean_v.restype = ctypes.c_float
    lib.ora_mean_v.argtypes = [i64, P]
    lib.ora_draw_message.restype = u32
    lib.ora_draw_message.argtypes = [u64, u32, u32, u64]
    lib.ora_tensor_means.restype = None
    lib.ora_tensor_means.argtypes = [i32, P, P, P]
    lib.ora_budget_expected.restype = i64
    lib.ora_budget_expected.argtypes = [i32, P, P, ctypes.c_float, ctypes.c_float]
    lib.ora_budget_c.restype = ctypes.c_float
    lib.ora_budget_c.argtypes = [i32, P, P, ctypes.c_float, i64]
    lib.ora_draw_tensor.restype = u32
    lib.ora_draw_tensor.argtypes = [u64, u32, u32, u64, i32]
    lib.ora_tensor_select.restype = i64
    lib.ora_tensor_select.argtypes = [i32, P, P, ctypes.c_float, ctypes.c_float, u64, u32, u32,
                                      u64, P]
    lib.ora_apply_tensors.restype = None
    lib.ora_apply_tensors.argtypes = [i32, i32, P, P, P, P, P, P, P, R, R, R, R]
    lib.ora_sim_grad.restype = None
    lib.ora_sim_grad.argtypes = [i64, P, P, P, P, u64, u32, u64, P]
    lib.ora_sim_loss.restype = ctypes.c_double
    lib.ora_sim_loss.argtypes = [i64, P, P, P]
    assert lib.ora_real_bytes() == (4 if real == "f32" else 8)
    return lib


def _load(real: str) -> ctypes.CDLL:
    with _LOCK:
        if real not in _LIBS:
            build()
            _LIBS[real] = load_library(lib_path(real), real)
        return _LIBS[real]


def _dtype(real: str):
    return np.float32 if real == "f32" else np.float64


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def coef(variant: int, alpha: float, tau: int, real: str = "f32", lib=None):
    """alpha(tau): alpha for ASGD, alpha / max(tau, 1) otherwise (Eq. 1, 7)."""
    return (lib or _load(real)).ora_coef(variant, alpha, tau)


def philox4x32_10(ctr, key, lib=None) -> list:
    """Philox4x32-10 block: four 32-bit words from a 4-word counter, 2-word key."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    o = np.zeros(4, dtype=np.uint32)
    (lib or _load("f32")).ora_philox4x32_10(_ptr(c), _ptr(k), _ptr(o))
    return [int(x) for x in o]


def draw(seed: int, client: int, push_no: int, p: int, lib=None) -> int:
    """24-bit uniform draw u_p of one parameter for one push."""
    return int((lib or _load("f32")).ora_draw(seed, client, push_no, p))


def decide(u: int, v: float, c: float, eps_b: float, lib=None) -> bool:
    """Eq. 9 in fp32: transmit iff u/2^24 < 1 / (1 + c / (v + eps_b))."""
    return bool((lib or _load("f32")).ora_decide(u, v, c, eps_b))


def select(g: np.ndarray, v: np.ndarray, c: float, eps_b: float, seed: int,
           client: int, push_no: int, lib=None):
    """B-FASGD send decision + compaction; returns (idx int32[m], val fp32[m])."""
    g = np.ascontiguousarray(g, dtype=np.float32)
    v = np.ascontiguousarray(v, dtype=np.float32)
    P = g.shape[0]
    idx = np.empty(max(P, 1), dtype=np.int32)
    val = np.empty(max(P, 1), dtype=np.float32)
    m = (lib or _load("f32")).ora_select(P, _ptr(g), _ptr(v), c, eps_b, seed, client, push_no,
                                _ptr(idx), _ptr(val))
    return idx[:m].copy(), val[:m].copy()


def draw_stream(seed: int, stream: int, client: int, n: int, p: int, lib=None) -> int:
    """24-bit draw of parameter p for a client's n-th transmission of a stream
    (0: push, 1: fetch)."""
    return int((lib or _load("f32")).ora_draw_stream(seed, stream, client, n, p))


def fetch_select(theta: np.ndarray, v: np.ndarray, c: float, eps_b: float, seed: int,
                 client: int, fetch_no: int, lib=None):
    """B-FASGD per-parameter fetch decision + compaction of theta; (idx, val)."""
    th = np.ascontiguousarray(theta, dtype=np.float32)
    v = np.ascontiguousarray(v, dtype=np.float32)
    P = th.shape[0]
    idx = np.empty(max(P, 1), dtype=np.int32)
    val = np.empty(max(P, 1), dtype=np.float32)
    m = (lib or _load("f32")).ora_fetch_select(P, _ptr(th), _ptr(v), c, eps_b, seed, client,
                                               fetch_no, _ptr(idx), _ptr(val))
    return idx[:m].copy(), val[:m].copy()


def fetch_apply(theta_client: np.ndarray, idx: np.ndarray, val: np.ndarray, lib=None):
    """Client side of a fetch: overwrite theta_client at idx with val (in place)."""
    assert theta_client.dtype == np.float32 and theta_client.flags["C_CONTIGUOUS"]
    i = np.ascontiguousarray(idx, dtype=np.int32)
    x = np.ascontiguousarray(val, dtype=np.float32)
    (lib or _load("f32")).ora_fetch_apply(_ptr(theta_client), i.shape[0], _ptr(i), _ptr(x))


def mean_v(v: np.ndarray, real: str = "f32", lib=None) -> float:
    """The per-message statistic of Sec. 2.3: mean of v over all parameters (fp32)."""
    vv = np.ascontiguousarray(v, dtype=_dtype(real))
    return float((lib or _load(real)).ora_mean_v(vv.shape[0], _ptr(vv)))


def draw_message(seed: int, stream: int, client: int, n: int, lib=None) -> int:
    """24-bit draw of a client's n-th push (stream 0) or fetch (stream 1) message."""
    return int((lib or _load("f32")).ora_draw_message(seed, stream, client, n))


def _sizes(sizes) -> np.ndarray:
    s = np.ascontiguousarray(sizes, dtype=np.int64)
    assert s.ndim == 1 and s.size >= 1 and (s >= 1).all()
    return s


def tensor_means(v: np.ndarray, sizes, real: str = "f32", lib=None) -> np.ndarray:
    """vbar_t: mean of v over each contiguous tensor (the exact sum divided by
    the tensor's size, rounded once to fp32)."""
    s = _sizes(sizes)
    vv = np.ascontiguousarray(v, dtype=_dtype(real))
    assert vv.shape[0] == int(s.sum())
    out = np.empty(s.size, dtype=np.float32)
    (lib or _load(real)).ora_tensor_means(s.size, _ptr(s), _ptr(vv), _ptr(out))
    return out


def budget_expected(sizes, vbar, eps_b: float, x: float, lib=None) -> int:
    """E(x) = sum_t floor(s_t fl(a_t / fl(a_t + x)) 2^32), a_t = fl(vbar_t + eps_b)."""
    s = _sizes(sizes)
    vb = np.ascontiguousarray(vbar, dtype=np.float32)
    return int((lib or _load("f32")).ora_budget_expected(s.size, _ptr(s), _ptr(vb), eps_b, x))


def budget_c(sizes, vbar, eps_b: float, budget: int, lib=None) -> float:
    """Smallest threshold c (non-negative float or +inf) with E(c) <= min(B, P) 2^32."""
    s = _sizes(sizes)
    vb = np.ascontiguousarray(vbar, dtype=np.float32)
    return float((lib or _load("f32")).ora_budget_c(s.size, _ptr(s), _ptr(vb), eps_b,
                                                     int(budget)))


def draw_tensor(seed: int, stream: int, client: int, n: int, t: int, lib=None) -> int:
    """24-bit draw of tensor t for a client's n-th push (stream 0) or fetch (stream 1)."""
    return int((lib or _load("f32")).ora_draw_tensor(seed, stream, client, n, t))


def tensor_select(sizes, vbar, c: float, eps_b: float, seed: int, stream: int, client: int,
                  n: int, lib=None):
    """Per-tensor Eq. 9 decisions at threshold c: (sent uint8[T], parameters sent)."""
    s = _sizes(sizes)
    vb = np.ascontiguousarray(vbar, dtype=np.float32)
    sent = np.zeros(s.size, dtype=np.uint8)
    m = (lib or _load("f32")).ora_tensor_select(s.size, _ptr(s), _ptr(vb), c, eps_b, seed,
                                                stream, client, n, _ptr(sent))
    return sent, int(m)


def sim_grad(theta, h, star, sigma, seed: int, client: int, n: int, lib=None) -> np.ndarray:
    """Stochastic gradient of the synthetic quadratic at theta (fp32[P])."""
    arrs = [np.ascontiguousarray(x, dtype=np.float32) for x in (theta, h, star, sigma)]
    g = np.empty_like(arrs[0])
    (lib or _load("f32")).ora_sim_grad(arrs[0].shape[0], *[_ptr(x) for x in arrs], seed, client,
                                       n, _ptr(g))
    return g


def sim_loss(theta, h, star, lib=None) -> float:
    """f(theta) = 1/2 sum h (theta - star)^2 (terms in fp32, sum in fp64)."""
    arrs = [np.ascontiguousarray(x, dtype=np.float32) for x in (theta, h, star)]
    return float((lib or _load("f32")).ora_sim_loss(arrs[0].shape[0], *[_ptr(x) for x in arrs]))


class OracleError(Exception):
    pass


class OracleServer:
    """The parameter server of Sections 2.1-2.3, one push at a time.

    State theta, n, b, v (REAL[P]; n = b = v = 0 at start), timestamp T = 0,
    and a FIFO of pushes.  ``apply_pending(K)`` pops the first K pushes in
    arrival order; push k sees the server timestamp T it finds, so its
    step-staleness is tau = T - j.
    """

    def __init__(self, P: int, lam: int, alpha: float, variant: int, real: str = "f32",
                 gamma: float = 0.95, beta: float = 0.95, eps: float = 1e-4,
                 c_push: float = 0.0, eps_b: float = 1e-8, seed: int = 0, lib=None):
        self.lib = lib or _load(real)
        self.real = real
        dt = _dtype(real)
        self.P, self.lam, self.alpha, self.variant = int(P), int(lam), float(alpha), int(variant)
        self.theta = np.zeros(P, dtype=dt)
        self.n = np.zeros(P, dtype=dt)
        self.b = np.zeros(P, dtype=dt)
        self.v = np.zeros(P, dtype=dt)
        self.T = 0
        self.fifo: list = []
        self.push_count = [0] * lam
        self.fetch_count = [0] * lam
        self.c_fetch = 0.0
        self.cache: dict = {}          # client -> most recent sent gradient (message pushes)
        self.message_log: list = []    # decisions of applied message pushes, in order
        self.sizes: np.ndarray | None = None   # tensor partition (per-tensor pushes)
        self.budget_log: list = []     # (sent, c, parameters sent) of applied budget pushes
        self.set_hparams(gamma, beta, eps, c_push, eps_b, seed)

    def set_hparams(self, gamma, beta, eps, c_push, eps_b, seed):
        # Hyper-parameters are fp32 at the boundary; the fp64 build widens them.
        f = lambda x: float(np.float32(x))
        self.gamma, self.beta, self.eps = f(gamma), f(beta), f(eps)
        self.c_push, self.eps_b, self.seed = f(c_push), f(eps_b), int(seed)

    def set_params(self, theta0: np.ndarray):
        self.theta[:] = theta0

    def push(self, client: int, j: int, g: np.ndarray):
        self._check(client, j)
        self.fifo.append(("dense", int(client), int(j), np.asarray(g, dtype=np.float32)))

    def push_message(self, client: int, j: int, g: np.ndarray):
        """Literal B-FASGD push (Sec. 2.3): decided when applied, against the
        mean of v at that moment; a dropped push re-applies the client's most
        recent sent gradient (zeros if it has none)."""
        self._check(client, j)
        self.fifo.append(("message", int(client), int(j), np.asarray(g, dtype=np.float32)))

    def fetch_message(self, client: int, theta_client: np.ndarray) -> bool:
        """Literal B-FASGD fetch: one decision with c_fetch against the mean of
        v; on success the client's copy becomes theta.  Returns the decision."""
        if not 0 <= client < self.lam:
            raise OracleError("client out of range")
        n = self.fetch_count[client]
        self.fetch_count[client] += 1
        u = draw_message(self.seed, 1, client, n)
        vbar = mean_v(self.v, self.real)
        ok = decide(u, vbar, self.c_fetch, self.eps_b)
        if ok:
            theta_client[:] = self.theta.astype(np.float32)
        return ok

    def set_tensors(self, sizes):
        """Partition the parameters into contiguous tensors (sizes sum to P)."""
        s = _sizes(sizes)
        if int(s.sum()) != self.P:
            raise OracleError("tensor sizes must sum to P")
        if self.fifo:
            raise OracleError("pushes are pending")
        self.sizes = s

    def _budget_decide(self, stream: int, client: int, n: int, budget: int):
        vbar = tensor_means(self.v, self.sizes, self.real)
        c = budget_c(self.sizes, vbar, self.eps_b, budget)
        sent, m = tensor_select(self.sizes, vbar, c, self.eps_b, self.seed, stream, client, n)
        return sent, c, m

    def push_budget(self, client: int, j: int, g: np.ndarray, budget: int):
        """Per-tensor B-FASGD push under a budget of `budget` expected
        parameters (decided when applied, against the server's v then)."""
        if self.sizes is None:
            raise OracleError("no tensor partition")
        if budget < 0:
            raise OracleError("budget must be >= 0")
        self._check(client, j)
        self.fifo.append(("budget", int(client), int(j),
                          (np.asarray(g, dtype=np.float32), int(budget))))

    def fetch_budget(self, client: int, theta_client: np.ndarray, budget: int):
        """Per-tensor B-FASGD fetch under a budget: the transmitted tensors of
        theta overwrite the client's copy.  Returns (sent, c, parameters sent)."""
        if self.sizes is None:
            raise OracleError("no tensor partition")
        if not 0 <= client < self.lam or budget < 0:
            raise OracleError("client or budget out of range")
        n = self.fetch_count[client]
        self.fetch_count[client] += 1
        sent, c, m = self._budget_decide(1, client, n, budget)
        off = np.concatenate([[0], np.cumsum(self.sizes)])
        for t in np.flatnonzero(sent):
            theta_client[off[t]:off[t + 1]] = self.theta[off[t]:off[t + 1]].astype(np.float32)
        return sent, c, m

    def push_sparse(self, client: int, j: int, idx: np.ndarray, val: np.ndarray):
        self._check(client, j)
        self.fifo.append(("sparse", int(client), int(j),
                          (np.ascontiguousarray(idx, dtype=np.int32),
                           np.ascontiguousarray(val, dtype=np.float32))))

    def _check(self, client, j):
        if not 0 <= client < self.lam:
            raise OracleError("client out of range")
        if not 0 <= j <= self.T:
            raise OracleError("timestamp out of range")

    def apply_pending(self, K: int):
        if K > len(self.fifo):
            raise OracleError("fewer pending pushes than K")
        for _ in range(K):
            kind, client, j, payload = self.fifo.pop(0)
            tau = self.T - j
            c = self.lib.ora_coef(self.variant, self.alpha, tau)
            if kind == "message":
                n = self.push_count[client]
                self.push_count[client] += 1
                u = draw_message(self.seed, 0, client, n)
                vbar = mean_v(self.v, self.real)
                sent = decide(u, vbar, self.c_push, self.eps_b)
                self.message_log.append(sent)
                if sent:
                    self.cache[client] = payload.copy()
                kind = "dense"
                payload = self.cache.get(client, np.zeros(self.P, np.float32))
            if kind == "budget":
                g, budget = payload
                n = self.push_count[client]
                self.push_count[client] += 1
                sent, cb, m = self._budget_decide(0, client, n, budget)
                self.budget_log.append((sent, cb, m))
                g = np.ascontiguousarray(g, dtype=np.float32)
                self.lib.ora_apply_tensors(self.variant, self.sizes.size, _ptr(self.sizes),
                                           _ptr(sent), _ptr(self.theta), _ptr(self.n),
                                           _ptr(self.b), _ptr(self.v), _ptr(g), c,
                                           self.gamma, self.beta, self.eps)
            elif kind == "dense":
                g = np.ascontiguousarray(payload, dtype=np.float32)
                self.lib.ora_apply_dense(self.variant, self.P, _ptr(self.theta), _ptr(self.n),
                                         _ptr(self.b), _ptr(self.v), _ptr(g), c,
                                         self.gamma, self.beta, self.eps)
            else:
                idx, val = payload
                rc = self.lib.ora_apply_sparse(self.variant, self.P, _ptr(self.theta),
                                               _ptr(self.n), _ptr(self.b), _ptr(self.v),
                                               idx.shape[0], _ptr(idx), _ptr(val), c,
                                               self.gamma, self.beta, self.eps)
                if rc != 0:
                    raise OracleError("bad sparse list")
            self.T += 1

    def select_compact(self, client: int, g: np.ndarray, v: np.ndarray | None = None):
        """B-FASGD push side for one client gradient; v defaults to the server's v."""
        if not 0 <= client < self.lam:
            raise OracleError("client out of range")
        vv = (self.v if v is None else v).astype(np.float32)
        out = select(g, vv, self.c_push, self.eps_b, self.seed, client,
                     self.push_count[client], lib=self.lib if self.real == "f32" else None)
        self.push_count[client] += 1
        return out

    def set_fetch_threshold(self, c_fetch: float):
        self.c_fetch = float(np.float32(c_fetch))

    def fetch_compact(self, client: int, v: np.ndarray | None = None):
        """B-FASGD fetch for one client: the kept (idx, theta[idx]) pairs."""
        if not 0 <= client < self.lam:
            raise OracleError("client out of range")
        vv = (self.v if v is None else v).astype(np.float32)
        out = fetch_select(self.theta.astype(np.float32), vv, self.c_fetch, self.eps_b,
                           self.seed, client, self.fetch_count[client],
                           lib=self.lib if self.real == "f32" else None)
        self.fetch_count[client] += 1
        return out

    def pull(self):
        return self.theta.copy(), self.T

    def state(self):
        return self.theta.copy(), self.n.copy(), self.b.copy(), self.v.copy(), self.T
