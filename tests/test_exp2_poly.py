"""The polynomial exponential of the attention kernels' softmax (no GPU):
its constants are the fitted minimax coefficients, its error bound holds,
and a float32 model of the kernel's bit manipulation reproduces 2^x over
the range the softmax feeds it, masked (-inf) scores included."""
import os
import re

import numpy as np

from paper_2609_32166_gb300 import exp2_poly

HERE = os.path.dirname(os.path.abspath(__file__))
PTX = os.path.join(HERE, "..", "paper_2609_32166_gb300", "csrc", "pf_ptx.cuh")


def kernel_constants():
    src = open(PTX).read()
    return np.array([float(re.search(r"kExp2C%d = ([0-9.eE+-]+)f;" % k, src).group(1))
                     for k in range(4)], dtype=np.float32)


def test_constants_are_the_fit():
    assert np.array_equal(kernel_constants(), exp2_poly.fit())


def test_error_bound():
    assert exp2_poly.max_relative_error(kernel_constants()) < 8e-5


def model(x):
    """float32 model of exp2_poly_x2: clamp, round by adding 1.5 * 2^23,
    Horner, exponent add."""
    c = kernel_constants()
    x = np.maximum(np.asarray(x, np.float32), np.float32(-126.0))
    t = (x + np.float32(12582912.0)).astype(np.float32)
    n = (t - np.float32(12582912.0)).astype(np.float32)
    f = (x - n).astype(np.float32)
    p = np.float32(c[3])
    for k in (2, 1, 0):
        p = (p * f + c[k]).astype(np.float32)
    bits = p.view(np.uint32) + (t.view(np.uint32) << np.uint32(23))
    return bits.astype(np.uint32).view(np.float32)


def test_model_matches_exp2_over_the_softmax_range():
    x = np.concatenate([np.linspace(-125.0, 8.0, 100001, dtype=np.float32),
                        np.array([0.0, -0.5, 0.5, 1.5, -1.5, 7.999], np.float32)])
    got = model(x).astype(np.float64)
    want = np.exp2(x.astype(np.float64))
    assert np.all(np.abs(got / want - 1.0) < 8e-5)


def test_masked_scores_give_zero_to_every_use():
    got = model(np.array([-np.inf, -1e30, -200.0, -126.0], np.float32))
    assert np.all(got >= 0) and np.all(got < 2.0 ** -125) and np.all(np.isfinite(got))
