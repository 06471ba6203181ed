"""The FMA-pipe exponential of the attention kernel, checked on the CPU.

The kernel evaluates part of the softmax exponentials as 2^n * p(f) with a
degree-3 polynomial instead of the MUFU ex2 instruction. This test reads the
coefficients from the kernel source and replays the same float32 steps with
NumPy: the relative error must stay far below the bf16 resolution of P, and
-inf / very negative arguments must give exactly 0.
"""
import os
import re

import numpy as np

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                   "paper_2608_20397_gb300", "csrc", "attention_kernels.cu")


def _coeffs():
    src = open(SRC).read()
    c = [float(re.search(rf"kExp2C{i} = ([0-9.eE+-]+)f;", src).group(1)) for i in range(4)]
    return [np.float32(x) for x in c]


def exp2_poly_f32(x):
    c0, c1, c2, c3 = _coeffs()
    x = np.asarray(x, np.float32)
    xc = np.maximum(x, np.float32(-125.0))
    M = np.float32(12582912.0)
    t = (xc + M).astype(np.float32)
    n = (t - M).astype(np.float32)
    f = (xc - n).astype(np.float32)
    p = (((c3 * f + c2) * f + c1) * f + c0).astype(np.float32)
    bits = p.view(np.int32) + (t.view(np.int32) << 23)
    y = bits.view(np.float32)
    return np.where(x < -125.0, np.float32(0.0), y)


def test_relative_error_over_the_softmax_range():
    x = np.concatenate([np.linspace(-125.0, 8.0, 400001), np.linspace(-1, 1, 100001)]).astype(np.float32)
    got = exp2_poly_f32(x).astype(np.float64)
    want = np.exp2(x.astype(np.float64))
    rel = np.abs(got / want - 1.0)
    assert rel.max() < 1e-4          # bf16 P resolves 2^-9 ~ 2e-3
    assert np.all(got > 0)


def test_masked_and_underflow_give_zero():
    x = np.array([-np.inf, -1e30, -125.5, -200.0], np.float32)
    assert np.all(exp2_poly_f32(x) == 0.0)
    assert exp2_poly_f32(np.array([0.0], np.float32))[0] == np.float32(_coeffs()[0])
