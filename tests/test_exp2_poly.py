"""The attention kernel's optional FMA-pipe exponential (exp2_poly_x2 in
csrc/tc_common.cuh), restated step by step in float32 on the host: its
relative error against the exact 2^x stays below the bound its comment states
(7.5e-5, under bf16's 2^-9 rounding of P) over the softmax's argument range."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def coefficients():
    src = open(os.path.join(ROOT, "paper_2609_30096_gb300", "csrc", "tc_common.cuh")).read()
    return [np.float32(float(re.search(rf"EXP2_C{i} = ([0-9.e+-]+)f", src).group(1)))
            for i in range(4)]


def exp2_poly(x):
    """The kernel's steps in float32: clamp, shifter rounding, degree-3 Horner in
    fused multiply-adds (emulated exactly in float64 then rounded), exponent add."""
    c0, c1, c2, c3 = coefficients()
    x = np.maximum(np.asarray(x, np.float32), np.float32(-126.0))
    sh = np.float32(12582912.0)
    j = (x + sh).astype(np.float32)
    f = (x - (j - sh).astype(np.float32)).astype(np.float32)
    fma = lambda a, b, c: (a.astype(np.float64) * b + c).astype(np.float32)
    p = fma(f, c3, c2)
    p = fma(p, f, c1)
    p = fma(p, f, c0)
    bits = p.view(np.uint32) + (j.view(np.uint32) << np.uint32(23))
    return bits.astype(np.uint32).view(np.float32)


def test_relative_error_bound_over_the_softmax_range():
    # normal results: x >= -125.5 (below, the exponent field underflows and the
    # value, under 2^-125, is only required to stay tiny and non-negative)
    x = np.concatenate([np.linspace(-125.5, 8.0, 2_000_001, dtype=np.float32),
                        np.float32([0.0, -0.5, 0.5, -1.5, 7.5, -125.5])])
    got = exp2_poly(x).astype(np.float64)
    ref = np.exp2(x.astype(np.float64))
    assert np.max(np.abs(got / ref - 1.0)) < 7.6e-5


def test_integer_arguments_and_clamp():
    n = np.arange(-125, 9, dtype=np.float32)
    got = exp2_poly(n).astype(np.float64)
    assert np.max(np.abs(got / np.exp2(n.astype(np.float64)) - 1.0)) < 7.6e-5
    assert exp2_poly(np.float32([-1000.0]))[0] == exp2_poly(np.float32([-126.0]))[0]
    tiny = exp2_poly(np.linspace(-1000.0, -125.5, 10001, dtype=np.float32))
    assert np.all(tiny >= 0.0) and np.all(tiny < 2.0 ** -125)
