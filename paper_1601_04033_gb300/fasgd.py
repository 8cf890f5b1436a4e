"""ctypes binding of include/fasgd.h (argument marshalling only).

Every function here forwards to the entry point of the same name in
libfasgd.so; all computation happens in the library's CUDA kernels.  The
library must have been built (``paper_1601_04033_gb300.build.build()`` or
``__graft_entry__.build()``); if it is missing, importing this module
raises -- there is no fallback.

``Server`` is a thin convenience wrapper over a handle that accepts torch
tensors (CUDA tensors for device arguments) and the current torch stream.
"""

from __future__ import annotations

import ctypes
import os

from . import build as _build

ASGD, SASGD, FASGD, FASGD_STD = 0, 1, 2, 3
OK, EINVAL, ERANGE, EAGAIN, ENOMEM, ECUDA, EDEVICE = 0, -1, -2, -3, -4, -5, -6
KMAX = 32
STATUS_NAMES = {OK: "OK", EINVAL: "EINVAL", ERANGE: "ERANGE", EAGAIN: "EAGAIN",
                ENOMEM: "ENOMEM", ECUDA: "ECUDA", EDEVICE: "EDEVICE"}

_p = ctypes.c_void_p
_i32, _i64, _u64, _f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_float

# name -> (restype, argtypes); the list mirrors include/fasgd.h one to one.
SIGNATURES = {
    "fasgd_create": (_i32, [ctypes.POINTER(_p), _i64, _i32, _f32, _i32]),
    "fasgd_destroy": (None, [_p]),
    "fasgd_set_hparams": (_i32, [_p, _f32, _f32, _f32, _f32, _f32, _u64]),
    "fasgd_set_stream": (_i32, [_p, _p]),
    "fasgd_set_exact": (_i32, [_p, _i32]),
    "fasgd_set_params": (_i32, [_p, _p]),
    "fasgd_push": (_i32, [_p, _i32, _i64, _p]),
    "fasgd_push_host": (_i32, [_p, _i32, _i64, _p]),
    "fasgd_push_sparse": (_i32, [_p, _i32, _i64, _p, _p, _p, _i64]),
    "fasgd_apply_pending": (_i32, [_p, _i32]),
    "bfasgd_select_compact": (_i32, [_p, _i32, _p, _p, _p, _p, _p]),
    "fasgd_pull": (_i32, [_p, _p, ctypes.POINTER(_i64)]),
    "fasgd_get_state": (_i32, [_p, _p, _p, _p, _p, ctypes.POINTER(_i64)]),
    "fasgd_set_state": (_i32, [_p, _p, _p, _p, _p, _i64]),
    "fasgd_get_push_counts": (_i32, [_p, _p]),
    "fasgd_set_push_counts": (_i32, [_p, _p]),
    "fasgd_sync": (_i32, [_p]),
    "fasgd_selftest_wait_expiry": (_i32, [_p]),
    "fasgd_selftest_fail_pass": (_i32, [_p, _i32]),
    "fasgd_timestamp": (_i64, [_p]),
    "fasgd_pending": (_i64, [_p]),
    "fasgd_kernel_launches": (_i64, [_p]),
    "bfasgd_fetch_compact": (_i32, [_p, _i32, _p, _p, _p, _p]),
    "fasgd_set_fetch_threshold": (_i32, [_p, _f32]),
    "bfasgd_fetch_apply": (_i32, [_i64, _p, _p, _p, _p, _i64, _p, _p]),
    "fasgd_get_fetch_counts": (_i32, [_p, _p]),
    "fasgd_set_fetch_counts": (_i32, [_p, _p]),
    "bfasgd_push_message": (_i32, [_p, _i32, _i64, _p, _p]),
    "bfasgd_fetch_message": (_i32, [_p, _i32, _p, _p]),
    "bfasgd_message_vbar": (_i32, [_p, _p]),
    "bfasgd_set_tensors": (_i32, [_p, _i32, _p]),
    "bfasgd_push_budget": (_i32, [_p, _i32, _i64, _p, _i64, _p, _p, _p]),
    "bfasgd_fetch_budget": (_i32, [_p, _i32, _p, _i64, _p, _p, _p]),
    "fasgd_sim_quadratic_grad": (_i32, [_i64, _p, _p, _p, _p, _u64, _i32, _u64, _p, _p]),
    "fasgd_sim_quadratic_loss": (_i32, [_i64, _p, _p, _p, _p, _p, _p]),
    "bfasgd_select_compact_noalloc": (_i32, [_i64, _p, _p, _f32, _f32, _u64, _i32, _u64,
                                             _p, _p, _p, _p]),
    "fasgd_last_error": (ctypes.c_char_p, [_p]),
}

NOALLOC_PMAX = 1 << 24
BFASGD_TMAX = 4096


def _load() -> ctypes.CDLL:
    path = _build.LIB
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build the CUDA library first "
                          "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


LIB = _load()
LIB_PATH = _build.LIB


class FasgdError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


# ---------------------------------------------------------------------------
# Raw entry points, same names and arguments as the C ABI (pointers as ints).
# ---------------------------------------------------------------------------
def fasgd_create(P: int, lam: int, alpha: float, variant: int):
    h = _p()
    rc = LIB.fasgd_create(ctypes.byref(h), P, lam, alpha, variant)
    return rc, h.value


def fasgd_destroy(h):
    LIB.fasgd_destroy(h)


def fasgd_set_hparams(h, gamma, beta, eps, c_push, eps_b, seed):
    return LIB.fasgd_set_hparams(h, gamma, beta, eps, c_push, eps_b, seed)


def fasgd_set_exact(h, exact):
    return LIB.fasgd_set_exact(h, exact)


def fasgd_set_stream(h, stream):
    return LIB.fasgd_set_stream(h, stream)


def fasgd_set_params(h, theta0):
    return LIB.fasgd_set_params(h, theta0)


def fasgd_push(h, client, timestamp, grad):
    return LIB.fasgd_push(h, client, timestamp, grad)


def fasgd_push_host(h, client, timestamp, grad_host):
    return LIB.fasgd_push_host(h, client, timestamp, grad_host)


def fasgd_push_sparse(h, client, timestamp, idx, val, n_dev, n_max):
    return LIB.fasgd_push_sparse(h, client, timestamp, idx, val, n_dev, n_max)


def fasgd_apply_pending(h, K):
    return LIB.fasgd_apply_pending(h, K)


def bfasgd_select_compact(h, client, grad, v, idx, val, n_dev):
    return LIB.bfasgd_select_compact(h, client, grad, v, idx, val, n_dev)


def bfasgd_fetch_compact(h, client, v, idx, val, n_dev):
    return LIB.bfasgd_fetch_compact(h, client, v, idx, val, n_dev)


def fasgd_set_fetch_threshold(h, c_fetch):
    return LIB.fasgd_set_fetch_threshold(h, c_fetch)


def bfasgd_fetch_apply(P, theta_client, idx, val, n_dev, n_max, stream, err_dev):
    return LIB.bfasgd_fetch_apply(P, theta_client, idx, val, n_dev, n_max, stream, err_dev)


def fasgd_get_fetch_counts(h, counts):
    return LIB.fasgd_get_fetch_counts(h, counts)


def fasgd_set_fetch_counts(h, counts):
    return LIB.fasgd_set_fetch_counts(h, counts)


def bfasgd_push_message(h, client, timestamp, grad, sent_dev):
    return LIB.bfasgd_push_message(h, client, timestamp, grad, sent_dev)


def bfasgd_fetch_message(h, client, theta_client, fetched_dev):
    return LIB.bfasgd_fetch_message(h, client, theta_client, fetched_dev)


def bfasgd_message_vbar(h, vbar_dev):
    return LIB.bfasgd_message_vbar(h, vbar_dev)


def bfasgd_set_tensors(h, T, sizes):
    return LIB.bfasgd_set_tensors(h, T, sizes)


def bfasgd_push_budget(h, client, timestamp, grad, budget, sent_dev, c_dev, count_dev):
    return LIB.bfasgd_push_budget(h, client, timestamp, grad, budget, sent_dev, c_dev, count_dev)


def bfasgd_fetch_budget(h, client, theta_client, budget, sent_dev, c_dev, count_dev):
    return LIB.bfasgd_fetch_budget(h, client, theta_client, budget, sent_dev, c_dev, count_dev)


def fasgd_sim_quadratic_grad(P, theta, h, star, sigma, seed, client, n, grad, stream):
    return LIB.fasgd_sim_quadratic_grad(P, theta, h, star, sigma, seed, client, n, grad, stream)


def fasgd_sim_quadratic_loss(P, theta, h, star, scratch, loss, stream):
    return LIB.fasgd_sim_quadratic_loss(P, theta, h, star, scratch, loss, stream)


def fasgd_pull(h, params):
    T = _i64()
    rc = LIB.fasgd_pull(h, params, ctypes.byref(T))
    return rc, T.value


def fasgd_get_state(h, theta, n, b, v):
    T = _i64()
    rc = LIB.fasgd_get_state(h, theta, n, b, v, ctypes.byref(T))
    return rc, T.value


def fasgd_set_state(h, theta, n, b, v, T):
    return LIB.fasgd_set_state(h, theta, n, b, v, T)


def fasgd_get_push_counts(h, counts):
    return LIB.fasgd_get_push_counts(h, counts)


def fasgd_set_push_counts(h, counts):
    return LIB.fasgd_set_push_counts(h, counts)


def fasgd_sync(h):
    return LIB.fasgd_sync(h)


def fasgd_selftest_wait_expiry(h):
    return LIB.fasgd_selftest_wait_expiry(h)


def fasgd_selftest_fail_pass(h, after):
    return LIB.fasgd_selftest_fail_pass(h, after)


def fasgd_timestamp(h):
    return LIB.fasgd_timestamp(h)


def fasgd_pending(h):
    return LIB.fasgd_pending(h)


def fasgd_kernel_launches(h):
    return LIB.fasgd_kernel_launches(h)


def bfasgd_select_compact_noalloc(P, grad, v, c, eps_b, seed, client, push_no, idx, val,
                                  n_dev, stream):
    return LIB.bfasgd_select_compact_noalloc(P, grad, v, c, eps_b, seed, client, push_no, idx,
                                             val, n_dev, stream)


def fasgd_last_error(h) -> str:
    s = LIB.fasgd_last_error(h)
    return s.decode() if s else ""


# ---------------------------------------------------------------------------
# Tensor-level wrapper
# ---------------------------------------------------------------------------
def _ptr(t) -> int | None:
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


def aligned_vectors(data, device="cuda"):
    """Copy a [R, P] array (numpy or torch) to the device as R fp32 vectors of
    length P whose starts are 16-byte aligned, as fasgd_push and
    bfasgd_select_compact require: rows are padded to a multiple of four
    floats inside one allocation.  Returns (backing tensor, list of views)."""
    import torch
    src = torch.as_tensor(data)
    R, P = src.shape
    pad = (P + 3) // 4 * 4
    buf = torch.empty((R, pad), dtype=torch.float32, device=device)
    buf[:, :P].copy_(src)
    return buf, [buf[r, :P] for r in range(R)]


def fetch_apply(theta_client, idx, val, n_dev=None, n_max=None, err_dev=None, stream=None):
    """Client side of a B-FASGD fetch (bfasgd_fetch_apply) on torch tensors."""
    import torch
    if n_max is None:
        n_max = idx.numel()
    s = stream if stream is not None else torch.cuda.current_stream()
    rc = bfasgd_fetch_apply(theta_client.numel(), _ptr(theta_client), _ptr(idx), _ptr(val),
                            _ptr(n_dev), n_max, s.cuda_stream, _ptr(err_dev))
    if rc != OK:
        raise FasgdError(rc, fasgd_last_error(None))


class Server:
    """One FASGD parameter server on the current CUDA device.

    Device arguments are torch CUDA tensors (fp32 / int32 / int64); the
    handle runs on torch's current stream at construction time unless a
    stream is given.
    """

    def __init__(self, P: int, lam: int, alpha: float, variant: int = FASGD, *,
                 gamma: float = 0.95, beta: float = 0.95, eps: float = 1e-4,
                 c_push: float = 0.0, eps_b: float = 1e-8, seed: int = 0, stream=None):
        import torch
        rc, h = fasgd_create(P, lam, alpha, variant)
        if rc != OK:
            raise FasgdError(rc, fasgd_last_error(None))
        self.h = h
        self.P, self.lam, self.variant = P, lam, variant
        self._check(fasgd_set_hparams(h, gamma, beta, eps, c_push, eps_b, seed))
        s = stream if stream is not None else torch.cuda.current_stream()
        self.stream = s
        self._check(fasgd_set_stream(h, s.cuda_stream))

    def _check(self, rc):
        if rc != OK:
            raise FasgdError(rc, fasgd_last_error(self.h))
        return rc

    def set_stream(self, stream):
        """Enqueue every later call on `stream` (a torch CUDA stream)."""
        self._check(fasgd_set_stream(self.h, stream.cuda_stream))
        self.stream = stream

    def close(self):
        if getattr(self, "h", None):
            fasgd_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- calls ---------------------------------------------------------------
    def set_hparams(self, gamma, beta, eps, c_push, eps_b, seed):
        self._check(fasgd_set_hparams(self.h, gamma, beta, eps, c_push, eps_b, seed))

    def set_exact(self, exact: bool):
        self._check(fasgd_set_exact(self.h, 1 if exact else 0))

    def set_params(self, theta0):
        self._check(fasgd_set_params(self.h, _ptr(theta0)))

    def push(self, client: int, timestamp: int, grad):
        self._check(fasgd_push(self.h, client, timestamp, _ptr(grad)))

    def push_host(self, client: int, timestamp: int, grad_host):
        self._check(fasgd_push_host(self.h, client, timestamp, _ptr(grad_host)))

    def push_sparse(self, client: int, timestamp: int, idx, val, n_dev=None, n_max=None):
        if n_max is None:
            n_max = idx.numel()
        self._check(fasgd_push_sparse(self.h, client, timestamp, _ptr(idx), _ptr(val),
                                      _ptr(n_dev), n_max))

    def apply_pending(self, K: int):
        self._check(fasgd_apply_pending(self.h, K))

    def select_compact(self, client: int, grad, idx, val, n_dev, v=None):
        self._check(bfasgd_select_compact(self.h, client, _ptr(grad), _ptr(v), _ptr(idx),
                                          _ptr(val), _ptr(n_dev)))

    def set_fetch_threshold(self, c_fetch: float):
        self._check(fasgd_set_fetch_threshold(self.h, c_fetch))

    def fetch_compact(self, client: int, idx, val, n_dev, v=None):
        self._check(bfasgd_fetch_compact(self.h, client, _ptr(v), _ptr(idx), _ptr(val),
                                         _ptr(n_dev)))

    def push_message(self, client: int, timestamp: int, grad, sent_dev=None):
        self._check(bfasgd_push_message(self.h, client, timestamp, _ptr(grad), _ptr(sent_dev)))

    def fetch_message(self, client: int, theta_client, fetched_dev=None):
        self._check(bfasgd_fetch_message(self.h, client, _ptr(theta_client), _ptr(fetched_dev)))

    def message_vbar(self, vbar_dev=None):
        """The per-message statistic (mean of v) now: written to vbar_dev if
        given (returns None), else returned as a float (synchronises)."""
        import torch
        out = vbar_dev if vbar_dev is not None else torch.empty(1, device="cuda")
        self._check(bfasgd_message_vbar(self.h, _ptr(out)))
        return None if vbar_dev is not None else float(out.item())

    def set_tensors(self, sizes):
        """Partition theta into contiguous tensors (sizes: ints summing to P)."""
        import numpy as np
        s = np.ascontiguousarray(sizes, dtype=np.int64)
        self._check(bfasgd_set_tensors(self.h, int(s.size), s.ctypes.data))

    def push_budget(self, client: int, timestamp: int, grad, budget: int, sent_dev=None,
                    c_dev=None, count_dev=None):
        """Per-tensor B-FASGD push under a budget of expected parameters."""
        self._check(bfasgd_push_budget(self.h, client, timestamp, _ptr(grad), int(budget),
                                       _ptr(sent_dev), _ptr(c_dev), _ptr(count_dev)))

    def fetch_budget(self, client: int, theta_client, budget: int, sent_dev=None, c_dev=None,
                     count_dev=None):
        """Per-tensor B-FASGD fetch into theta_client under a budget."""
        self._check(bfasgd_fetch_budget(self.h, client, _ptr(theta_client), int(budget),
                                        _ptr(sent_dev), _ptr(c_dev), _ptr(count_dev)))

    def fetch_counts(self):
        import numpy as np
        out = np.zeros(self.lam, dtype=np.uint64)
        self._check(fasgd_get_fetch_counts(self.h, out.ctypes.data))
        return out

    def pull(self, params=None) -> int:
        rc, T = fasgd_pull(self.h, _ptr(params))
        self._check(rc)
        return T

    def get_state(self, theta=None, n=None, b=None, v=None) -> int:
        rc, T = fasgd_get_state(self.h, _ptr(theta), _ptr(n), _ptr(b), _ptr(v))
        self._check(rc)
        return T

    def set_state(self, theta, n, b, v, T: int):
        self._check(fasgd_set_state(self.h, _ptr(theta), _ptr(n), _ptr(b), _ptr(v), T))

    def push_counts(self):
        import numpy as np
        out = np.zeros(self.lam, dtype=np.uint64)
        self._check(fasgd_get_push_counts(self.h, out.ctypes.data))
        return out

    def set_push_counts(self, counts):
        import numpy as np
        c = np.ascontiguousarray(counts, dtype=np.uint64)
        self._check(fasgd_set_push_counts(self.h, c.ctypes.data))

    def sync(self):
        self._check(fasgd_sync(self.h))

    def selftest_wait_expiry(self):
        """Enqueue the pipeline-wait expiry self-test (the next sync reports EDEVICE)."""
        self._check(fasgd_selftest_wait_expiry(self.h))

    def selftest_fail_pass(self, after: int):
        """Make the pass of apply_pending `after` passes from now report a launch failure."""
        self._check(fasgd_selftest_fail_pass(self.h, after))

    @property
    def T(self) -> int:
        return fasgd_timestamp(self.h)

    @property
    def pending(self) -> int:
        return fasgd_pending(self.h)

    @property
    def launches(self) -> int:
        return fasgd_kernel_launches(self.h)
