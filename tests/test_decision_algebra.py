"""The CUDA select kernel decides Eq. 9 as err < fl(A - prod) (prod = fl(u d),
err = u d - prod exactly, A = a 2^24); the oracle uses a different exact
form.  Check on the CPU, with exact rationals, that the kernel's form equals
the exact predicate u d < A, including at and next to the threshold."""

from fractions import Fraction

import numpy as np


def kernel_form(u, a, d):
    uf = np.float32(u)
    prod = np.float32(uf * d)                                   # fl(u d)
    err = float(Fraction(int(u)) * Fraction(float(d)) - Fraction(float(prod)))  # exact fma
    A = np.float32(a * np.float32(16777216.0))
    return err < float(np.float32(A - prod))


def exact(u, a, d):
    return Fraction(int(u)) * Fraction(float(d)) < Fraction(float(a)) * (1 << 24)


def test_kernel_decision_form_is_exact():
    rng = np.random.default_rng(17)
    n = 0
    for _ in range(20000):
        a = np.float32(10 ** rng.uniform(-6, 4))
        c = np.float32(10 ** rng.uniform(-6, 4)) if rng.random() < 0.95 else np.float32(0)
        d = np.float32(a + c)
        t = float(a) * 2 ** 24 / float(d)
        if rng.random() < 0.7:
            u = int(np.clip(round(t) + int(rng.integers(-2, 3)), 0, 2 ** 24 - 1))
        else:
            u = int(rng.integers(0, 2 ** 24))
        assert kernel_form(u, a, d) == exact(u, a, d), (u, a, c)
        n += 1
    # exact ties: a = 2^k, d = 2^m
    for k in range(-4, 5):
        for m in range(k, k + 8):
            a, d = np.float32(2.0 ** k), np.float32(2.0 ** m)
            u = int(2 ** 24 * 2.0 ** (k - m))
            if 1 <= u < 2 ** 24:
                assert kernel_form(u, a, d) is False and exact(u, a, d) is False
                assert kernel_form(u - 1, a, d) is True
    assert n == 20000
