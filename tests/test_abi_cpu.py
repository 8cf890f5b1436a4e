"""The C-ABI library on a machine without a GPU: it builds, loads, exports
every entry point include/fasgd.h declares, and rejects bad arguments on the
host before touching the device."""

import ctypes
import os
import re

import pytest

from paper_1601_04033_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "fasgd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"FASGD_API\s+[\w\s\*]+?\b((?:b?fasgd)_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def binding():
    build.build()
    from paper_1601_04033_gb300 import fasgd
    return fasgd


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("fasgd_create", "fasgd_push", "fasgd_apply_pending",
                     "bfasgd_select_compact", "fasgd_pull", "fasgd_destroy"):
        assert required in names
    assert len(names) >= 20


def test_library_exports_every_declared_symbol(binding):
    lib = ctypes.CDLL(binding.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
    # The binding mirrors the header one to one.
    assert sorted(binding.SIGNATURES) == declared_functions()
    for name in declared_functions():
        assert callable(getattr(binding, name)), name


def test_only_the_abi_is_exported(binding):
    out = os.popen(f"nm -D --defined-only {binding.LIB_PATH}").read().split("\n")
    syms = sorted(line.split()[-1] for line in out if line.strip())
    assert syms == declared_functions()


def test_host_side_argument_checks(binding):
    f = binding
    # No device is touched before these are rejected.
    for P, lam, alpha, var in ((0, 4, 0.1, 2), (-5, 4, 0.1, 2), (1 << 31, 4, 0.1, 2),
                               (10, 0, 0.1, 2), (10, 1 << 21, 0.1, 2),
                               (10, 4, float("nan"), 2), (10, 4, float("inf"), 0),
                               (10, 4, 0.1, 4), (10, 4, 0.1, -1)):
        rc, h = f.fasgd_create(P, lam, alpha, var)
        assert rc == f.EINVAL and h is None, (P, lam, alpha, var)
        assert f.fasgd_last_error(None)
    assert f.LIB.fasgd_create(None, 10, 4, 0.1, 2) == f.EINVAL
    # A NULL handle is rejected by every call.
    assert f.fasgd_push(None, 0, 0, 16) == f.EINVAL
    assert f.fasgd_apply_pending(None, 1) == f.EINVAL
    assert f.bfasgd_select_compact(None, 0, 16, None, 16, 16, 16) == f.EINVAL
    assert f.fasgd_pull(None, None)[0] == f.EINVAL
    assert f.fasgd_sync(None) == f.EINVAL
    assert f.fasgd_timestamp(None) == -1 and f.fasgd_pending(None) == -1
    f.fasgd_destroy(None)


HANDLELESS = {"bfasgd_fetch_apply", "fasgd_sim_quadratic_grad", "fasgd_sim_quadratic_loss",
              "bfasgd_select_compact_noalloc", "fasgd_last_error", "fasgd_destroy",
              "fasgd_create"}


def test_every_handle_call_rejects_a_null_handle(binding):
    """Every entry point that takes a handle returns EINVAL (or -1 for the
    introspection calls) for NULL, before it reads any other argument."""
    f = binding
    for name, (res, argtypes) in f.SIGNATURES.items():
        if name in HANDLELESS:
            continue
        args = [None if t in (ctypes.c_void_p,) or hasattr(t, "contents") or
                t.__name__.startswith("LP_") else 0 for t in argtypes]
        rc = getattr(f.LIB, name)(*args)
        if res is ctypes.c_int64:
            assert rc == -1, name
        else:
            assert rc == f.EINVAL, name


def test_handleless_calls_check_their_arguments_on_the_host(binding):
    f = binding
    L = f.LIB
    a16, a4 = 1 << 12, (1 << 12) + 4      # never dereferenced: rejected or a no-op first
    # bfasgd_select_compact_noalloc(P, grad, v, c, eps_b, seed, client, push_no, idx, val, n, stream)
    good = [1000, a16, a16, 1.0, 1e-8, 7, 0, 0, a16, a16, a16 + 64, None]
    for k, bad in ((0, 0), (0, f.NOALLOC_PMAX + 1), (6, -1), (1, None), (1, a4), (2, None),
                   (3, -1.0), (3, float("nan")), (4, float("inf")), (4, -1.0), (8, None),
                   (9, None), (10, None), (10, a4)):
        args = list(good)
        args[k] = bad
        assert L.bfasgd_select_compact_noalloc(*args) == f.EINVAL, (k, bad)
        assert f.fasgd_last_error(None)
    # bfasgd_fetch_apply(P, theta, idx, val, n_dev, n_max, stream, err)
    good = [1000, a16, a16, a16, None, 0, None, None]
    assert L.bfasgd_fetch_apply(*good) == f.OK       # nothing to apply: no device work
    for k, bad in ((0, 0), (0, 1 << 31), (1, None), (5, -1), (5, 1001), (4, a4), (7, a4 + 2)):
        args = list(good)
        args[k] = bad
        assert L.bfasgd_fetch_apply(*args) == f.EINVAL, (k, bad)
    args = list(good)
    args[5] = 10                                      # entries but no lists
    args[2] = None
    assert L.bfasgd_fetch_apply(*args) == f.EINVAL
    # fasgd_sim_quadratic_grad(P, theta, h, star, sigma, seed, client, n, grad, stream)
    good = [1000, a16, a16, a16, a16, 1, 0, 0, a16, None]
    for k, bad in ((0, 0), (6, -1), (6, 1 << 30), (1, None), (2, a4), (4, None), (8, None)):
        args = list(good)
        args[k] = bad
        assert L.fasgd_sim_quadratic_grad(*args) == f.EINVAL, (k, bad)
    # fasgd_sim_quadratic_loss(P, theta, h, star, scratch, loss, stream)
    good = [1000, a16, a16, a16, a16, a16 + 64, None]
    for k, bad in ((0, 0), (1, None), (4, None), (4, a4), (5, None), (5, a4)):
        args = list(good)
        args[k] = bad
        assert L.fasgd_sim_quadratic_loss(*args) == f.EINVAL, (k, bad)


def test_c_callers_compile_and_link():
    """The header is plain C: the C timing driver of the ABI (abi_latency.c)
    compiles as C11 and links against the library."""
    exe = build.build_latency_driver(force=True)
    assert os.path.exists(exe) and os.access(exe, os.X_OK)
