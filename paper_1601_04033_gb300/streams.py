"""Seeded synthetic workloads for the FASGD parameter-server path.

This module only draws random inputs; it holds none of the method's
arithmetic (no moving averages, no step, no send decision).  Both the CUDA
path and the CPU oracle consume exactly the arrays made here, so the two
sides always see bit-identical inputs.

What is drawn, per workload (paper Section 4 uses MNIST and an MLP; neither
is available here, so these synthetic streams stand in for the clients'
gradients):

* theta0_p ~ N(0, 0.01^2)                         initial parameters
* m_p ~ N(0, 1e-3^2), s_p ~ log-uniform[lo, hi]   per-parameter gradient mean / spread
* pool slot r: grad_r = m + s * z_r, z_r ~ N(0,1) one full gradient vector per slot
* client of push t: t mod lambda                  round-robin arrival
* delay d_t from the workload's staleness law     (uniform / Poisson / geometric / Pareto)
* pool slot of push t: the K slots of one batch are distinct

The timestamp a push carries follows the protocol of Section 2.1: a client
pushes a gradient computed on parameters with timestamp j <= i, where i is
the server timestamp at the moment of the push.  Pushes are made in batches
of K against the server timestamp T_b = b*K before batch b is applied, and
push t carries j_t = T_b - min(d_t, T_b).
"""

from __future__ import annotations

import dataclasses
import math

import numpy as np

ASGD, SASGD, FASGD, FASGD_STD = 0, 1, 2, 3
VARIANT_NAMES = {ASGD: "asgd", SASGD: "sasgd", FASGD: "fasgd", FASGD_STD: "fasgd-std"}

# Sub-stream tags: each component gets its own PCG64 stream keyed by
# (seed, tag[, slot]) so that any one can be regenerated alone.
_TAG_THETA0, _TAG_MEAN, _TAG_SPREAD, _TAG_POOL, _TAG_DELAY, _TAG_SLOT = range(6)


def _rng(*key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(list(key)))


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload (sizes, staleness law, seed)."""

    name: str
    P: int                 # number of fp32 parameters
    lam: int               # number of clients (lambda)
    pushes: int            # pushes in the whole stream
    alpha: float           # master learning rate
    K: int                 # pending pushes fused into one server pass
    variants: tuple        # which update rules this workload exercises
    delay: str             # staleness law name, see delays()
    seed: int
    s_lo: float = 1e-4     # log-uniform range of the per-parameter spread s_p
    s_hi: float = 1e-1
    R: int = 16            # gradient pool slots (>= 2K)
    send_frac: float | None = None   # B-FASGD target send fraction, None = dense
    tensors: int = 0       # per-tensor B-FASGD: tensors in the partition (0: not used)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads the path is specified on.
WORKLOADS = {
    "fasgd-7850": Workload("fasgd-7850", 7_850, 4, 200, 0.01, 1,
                           (ASGD, SASGD, FASGD), "uniform4", 0),
    "fasgd-1.29m": Workload("fasgd-1.29m", 1_290_510, 32, 10_000, 0.005, 1,
                            (ASGD, SASGD, FASGD), "poisson4", 1),
    "fasgd-25m-k8": Workload("fasgd-25m-k8", 25_000_000, 128, 20_000, 0.001, 8,
                             (FASGD,), "geometric0.05", 2),
    "bfasgd-25m": Workload("bfasgd-25m", 25_000_000, 64, 10_000, 0.001, 1,
                           (FASGD,), "poisson8", 3, send_frac=0.20),
    # The paper's literal B-FASGD (one decision per message) on the 25M shape.
    "bfasgd-message-25m": Workload("bfasgd-message-25m", 25_000_000, 64, 10_000, 0.001, 1,
                                   (FASGD,), "poisson8", 3, send_frac=0.20),
    # Per-tensor B-FASGD with a bandwidth budget on the 25M shape: 160 tensors.
    "bfasgd-tensor-25m": Workload("bfasgd-tensor-25m", 25_000_000, 64, 10_000, 0.001, 1,
                                  (FASGD,), "poisson8", 3, send_frac=0.20, tensors=160),
    "fasgd-268m-k16": Workload("fasgd-268m-k16", 268_435_456, 256, 2_000, 0.001, 16,
                               (FASGD,), "pareto1.5", 4, s_lo=1e-5, s_hi=1.0, R=32,
                               send_frac=0.20),
    # Per-parameter B-FASGD exchanges on the 2^28 shape.
    "bfasgd-268m": Workload("bfasgd-268m", 268_435_456, 256, 2_000, 0.001, 1,
                            (FASGD,), "pareto1.5", 4, s_lo=1e-5, s_hi=1.0, R=32,
                            send_frac=0.20),
}


def theta0(w: Workload, P: int | None = None) -> np.ndarray:
    """Initial parameters, N(0, 0.01^2), fp32[P]."""
    P = w.P if P is None else P
    return (_rng(w.seed, _TAG_THETA0).standard_normal(P, dtype=np.float32)
            * np.float32(0.01))


def grad_model(w: Workload, P: int | None = None):
    """Per-parameter gradient mean m_p and spread s_p (fp32[P] each)."""
    P = w.P if P is None else P
    m = (_rng(w.seed, _TAG_MEAN).standard_normal(P, dtype=np.float32)
         * np.float32(1e-3))
    lo, hi = math.log(w.s_lo), math.log(w.s_hi)
    s = np.exp(_rng(w.seed, _TAG_SPREAD).uniform(lo, hi, P)).astype(np.float32)
    if w.tensors and P >= w.tensors:
        # Layer structure: each tensor's spreads share a scale, log-uniform
        # over two decades, so the per-tensor statistics differ.
        sizes = tensor_sizes(w.seed, P, w.tensors)
        scale = np.exp(_rng(w.seed, _TAG_TENSORS, 0).uniform(math.log(0.1), math.log(10.0),
                                                               w.tensors))
        s *= np.repeat(scale.astype(np.float32), sizes)
    return m, s


def pool_slot(w: Workload, r: int, m: np.ndarray, s: np.ndarray) -> np.ndarray:
    """Gradient vector of pool slot r: m + s * z_r (fp32 arithmetic)."""
    z = _rng(w.seed, _TAG_POOL, r).standard_normal(m.shape[0], dtype=np.float32)
    z *= s
    z += m
    return z


def gradient_pool(w: Workload, P: int | None = None, R: int | None = None,
                  threads: int = 16) -> np.ndarray:
    """All R pool slots as one fp32[R, P] array (slots drawn in parallel)."""
    import concurrent.futures
    P = w.P if P is None else P
    R = w.R if R is None else R
    m, s = grad_model(w, P)
    out = np.empty((R, P), dtype=np.float32)

    def fill(r):
        out[r] = pool_slot(w, r, m, s)

    with concurrent.futures.ThreadPoolExecutor(max_workers=max(1, min(threads, R))) as ex:
        list(ex.map(fill, range(R)))
    return out


def delays(w: Workload, n: int) -> np.ndarray:
    """Per-push staleness draws d_t (int64[n]) for the workload's law."""
    g = _rng(w.seed, _TAG_DELAY)
    if w.delay == "uniform4":            # U{0..3}
        d = g.integers(0, 4, n)
    elif w.delay == "poisson4":
        d = g.poisson(4.0, n)
    elif w.delay == "poisson8":
        d = g.poisson(8.0, n)
    elif w.delay == "geometric0.05":     # failures before the first success, {0,1,...}
        d = np.minimum(g.geometric(0.05, n) - 1, 512)
    elif w.delay == "pareto1.5":         # floor of a Lomax(1.5) draw (Pareto, scale 1, shifted to 0)
        d = np.minimum(np.floor(g.pareto(1.5, n)), 4096)
    else:
        raise ValueError(f"unknown delay law {w.delay!r}")
    return d.astype(np.int64)


def slots(w: Workload, n: int) -> np.ndarray:
    """Pool slot of each push; the K slots inside one batch are distinct."""
    if w.R < w.K:
        raise ValueError("pool smaller than one batch")
    g = _rng(w.seed, _TAG_SLOT)
    nb = -(-n // w.K)
    out = np.empty(nb * w.K, dtype=np.int64)
    for b in range(nb):
        out[b * w.K:(b + 1) * w.K] = g.choice(w.R, w.K, replace=False)
    return out[:n]


def clients(w: Workload, n: int) -> np.ndarray:
    """Round-robin client ids, t mod lambda."""
    return (np.arange(n, dtype=np.int64) % w.lam).astype(np.int32)


def timestamps(w: Workload, n: int, K: int | None = None) -> np.ndarray:
    """Timestamp j_t carried by push t when pushes arrive in batches of K.

    Batch b is pushed while the server timestamp is T_b = b*K and is then
    applied as a whole; push t of that batch carries j_t = T_b - min(d_t, T_b).
    """
    K = w.K if K is None else K
    d = delays(w, n)
    Tb = (np.arange(n, dtype=np.int64) // K) * K
    return Tb - np.minimum(d, Tb)


@dataclasses.dataclass
class PushStream:
    """The first n pushes of a workload: client, timestamp and pool slot."""

    client: np.ndarray
    j: np.ndarray
    slot: np.ndarray
    K: int

    @property
    def n(self) -> int:
        return int(self.client.shape[0])

    def batch(self, b: int):
        """(clients, timestamps, slots) of batch b."""
        s = slice(b * self.K, (b + 1) * self.K)
        return self.client[s], self.j[s], self.slot[s]


def push_stream(w: Workload, n: int | None = None, K: int | None = None) -> PushStream:
    n = w.pushes if n is None else n
    K = w.K if K is None else K
    w2 = w if K == w.K else w.replace(K=K)
    return PushStream(clients(w2, n), timestamps(w2, n, K), slots(w2, n), K)


def sample_indices(P: int, count: int, seed: int = 12345) -> np.ndarray:
    """Sorted distinct parameter indices for sampled checks at full size.

    Always includes the first and last four indices (ragged tail)."""
    g = _rng(seed, 99, P)
    count = min(count, P)
    pick = g.choice(P, count, replace=False)
    edge = np.array([0, 1, 2, 3, P - 4, P - 3, P - 2, P - 1], dtype=np.int64)
    edge = edge[(edge >= 0) & (edge < P)]
    return np.unique(np.concatenate([pick.astype(np.int64), edge]))


_TAG_VSNAP = 6


def client_v_snapshot(w: Workload, client: int, P: int | None = None,
                      lo: float = 1.0, hi: float = 100.0) -> np.ndarray:
    """A client's copy of the server statistic v (fp32[P], log-uniform[lo, hi]).

    B-FASGD clients decide with the v they last fetched from the server; a
    drawn snapshot stands in for it where both sides of a comparison must
    decide on identical inputs."""
    P = w.P if P is None else P
    u = _rng(w.seed, _TAG_VSNAP, client).uniform(math.log(lo), math.log(hi), P)
    return np.exp(u).astype(np.float32)


_TAG_OBJ_H, _TAG_OBJ_STAR, _TAG_OBJ_SIGMA, _TAG_DISPATCH = 7, 8, 9, 10


def quadratic_objective(seed: int, P: int, h_lo: float = 1e-2, h_hi: float = 10.0,
                        sigma_lo: float = 1e-3, sigma_hi: float = 1e-1, noise: str = "independent",
                        tensors=None):
    """A synthetic separable quadratic for the closed-loop simulation:
    curvatures h_p log-uniform[h_lo, h_hi], minimiser star_p ~ N(0, 0.1^2),
    gradient-noise scales sigma_p log-uniform[sigma_lo, sigma_hi] (fp32[P] each;
    noise="fisher" instead ties the noise to the curvature, sigma_p =
    0.03 sqrt(h_p), as when the gradient covariance tracks the Hessian).
    The spread of h makes a single learning rate a compromise across
    parameters, as in a real network.  tensors (sizes of a partition of P):
    each tensor's curvatures are also scaled by a common factor, log-uniform
    over [0.1, 10], so that the tensors' statistics differ as layers do."""
    h = np.exp(_rng(seed, _TAG_OBJ_H).uniform(math.log(h_lo), math.log(h_hi), P)).astype(np.float32)
    if tensors is not None:
        sizes = np.asarray(tensors, dtype=np.int64)
        assert int(sizes.sum()) == P
        f = np.exp(_rng(seed, _TAG_OBJ_H, 1).uniform(math.log(0.1), math.log(10.0), sizes.size))
        h = (h * np.repeat(f.astype(np.float32), sizes)).astype(np.float32)
    star = (_rng(seed, _TAG_OBJ_STAR).standard_normal(P, dtype=np.float32) * np.float32(0.1))
    if noise == "fisher":
        sigma = (np.float32(0.03) * np.sqrt(h)).astype(np.float32)
    else:
        sigma = np.exp(_rng(seed, _TAG_OBJ_SIGMA).uniform(math.log(sigma_lo), math.log(sigma_hi),
                                                          P)).astype(np.float32)
    return h, star, sigma


_TAG_TENSORS = 11


def tensor_sizes(seed: int, P: int, T: int) -> np.ndarray:
    """A partition of P parameters into T contiguous tensors with the size mix
    of a layered network: alternating weight tensors (relative sizes
    log-uniform over three decades) and vector tensors (biases / scales,
    log-uniform in [16, 4096] parameters, at most a quarter of P in all).
    P = 7,850 with T = 2 is the paper's softmax-regression model on 28x28
    inputs and 10 classes (784 x 10 weights, then 10 biases).  int64[T]."""
    if T < 1 or P < T:
        raise ValueError("need 1 <= T <= P")
    if T == 1:
        return np.array([P], np.int64)
    if P == 7_850 and T == 2:
        return np.array([7_840, 10], np.int64)
    g = _rng(seed, _TAG_TENSORS, T)
    n_vec = T // 2
    n_mat = T - n_vec
    vec = np.exp(g.uniform(math.log(16), math.log(4096), n_vec))
    vec = np.maximum(1, np.floor(vec * min(1.0, (P / 4) / vec.sum()))).astype(np.int64)
    rest = P - int(vec.sum())
    w = np.exp(g.uniform(0.0, math.log(1000.0), n_mat))
    mat = np.maximum(1, np.floor(w / w.sum() * (rest - n_mat))).astype(np.int64)
    mat[int(np.argmax(mat))] += rest - int(mat.sum())
    out = np.empty(T, np.int64)
    out[0::2] = mat
    out[1::2] = vec
    assert out.min() >= 1 and int(out.sum()) == P
    return out


def dispatch_schedule(seed: int, lam: int, n_batches: int, K: int = 1, rho: float = 1.0):
    """Which clients push in each batch of K (distinct within a batch: a client
    waits for the server's reply before it pushes again, Sec. 3).  Selection
    weights start at 1; a selected client's weight is multiplied by rho and
    every other weight by 1/rho, capped at 1 (rho = 1: uniform choice)."""
    if K > lam:
        raise ValueError("K clients per batch need lambda >= K")
    g = _rng(seed, _TAG_DISPATCH)
    w = np.ones(lam)
    out = np.empty((n_batches, K), dtype=np.int32)
    for b in range(n_batches):
        pick = g.choice(lam, K, replace=False, p=w / w.sum())
        out[b] = pick
        if rho != 1.0:
            mask = np.zeros(lam, bool)
            mask[pick] = True
            w[mask] *= rho
            w[~mask] = np.minimum(1.0, w[~mask] / rho)
    return out
