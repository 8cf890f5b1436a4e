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
