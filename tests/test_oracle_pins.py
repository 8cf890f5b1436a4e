"""The CPU oracle against what the paper and the mathematics fix (no GPU)."""

import pytest

import pins


@pytest.fixture(scope="module")
def libs():
    return pins.real_libs()


@pytest.mark.parametrize("check", pins.ALL_CHECKS, ids=lambda f: f.__name__)
def test_pin(libs, check):
    check(libs)
