"""Coefficients of the degree-3 polynomial for 2^f on [-1/2, 1/2] that the
attention kernels use to take part of their exponentials off the
special-function unit (exp2_poly_x2 in csrc/pf_ptx.cuh).

The fit minimises the maximum relative error |p(f) / 2^f - 1| by Lawson's
algorithm: weighted least squares on a dense grid, each weight multiplied by
its point's current error until the weights settle on the extremal points.
Run as a script to print the coefficients the kernel holds.
"""
from __future__ import annotations

import numpy as np


def fit(degree: int = 3, points: int = 20001, iterations: int = 200) -> np.ndarray:
    f = np.linspace(-0.5, 0.5, points)
    y = np.exp2(f)
    A = np.stack([f ** k for k in range(degree + 1)], 1) / y[:, None]
    w = np.full(points, 1.0 / points)
    c = None
    for _ in range(iterations):
        W = np.sqrt(w)
        c, *_ = np.linalg.lstsq(A * W[:, None], W, rcond=None)
        r = np.abs(A @ c - 1.0)
        w = w * r
        w /= w.sum()
    return c.astype(np.float32)


def max_relative_error(c32: np.ndarray, points: int = 200001) -> float:
    """Worst relative error of the float32 Horner evaluation of c32 against
    2^f over [-1/2, 1/2] (float64 reference)."""
    f = np.linspace(-0.5, 0.5, points).astype(np.float32)
    p = np.full_like(f, c32[-1])
    for k in range(len(c32) - 2, -1, -1):
        p = (p * f + c32[k]).astype(np.float32)
    return float(np.abs(p.astype(np.float64) / np.exp2(f.astype(np.float64)) - 1.0).max())


if __name__ == "__main__":
    c = fit()
    print([repr(float(x)) for x in c], max_relative_error(c))
