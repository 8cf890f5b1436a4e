"""Choose the B-FASGD threshold c for a target send fraction.

Under Eq. 9 parameter p is sent with probability t_p = a_p / (a_p + c),
a_p = v_p + eps_b.  The expected fraction sent, mean_p t_p, falls
monotonically in c, so bisection on c finds the value that meets a target
fraction (e.g. 0.20 for a 5x cut of push bandwidth) for a given v.
"""

from __future__ import annotations

import numpy as np


def expected_send_fraction(v: np.ndarray, c: float, eps_b: float) -> float:
    a = np.asarray(v, dtype=np.float64) + eps_b
    return float(np.mean(a / (a + c)))


def calibrate_c(v: np.ndarray, target: float, eps_b: float = 1e-8, iters: int = 80) -> float:
    """c >= 0 with expected_send_fraction(v, c) = target (0 < target <= 1)."""
    if not 0.0 < target <= 1.0:
        raise ValueError("target must be in (0, 1]")
    if target == 1.0:
        return 0.0
    v = np.asarray(v, dtype=np.float64)
    lo, hi = 0.0, 1.0
    while expected_send_fraction(v, hi, eps_b) > target:
        hi *= 2.0
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if expected_send_fraction(v, mid, eps_b) > target:
            lo = mid
        else:
            hi = mid
    return float(np.float32(0.5 * (lo + hi)))
