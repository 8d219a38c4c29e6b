"""Pins of the oracle's chained epilogue: a linear whose output is the next
per-channel quantized linear's input writes that layer's codes directly
(fc1 -> ReLU -> fc2; Section 3.2's fusion carried to the fc1 epilogue)."""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from test_oracle_pins import frac_to_f32


@pytest.mark.parametrize("relu", [False, True])
def test_epilogue_quantize_exact_rounding(relu):
    """Every fp32 step evaluated as an exact rational and rounded once."""
    rng = np.random.default_rng(3)
    M, N = 6, 9
    acc = rng.integers(-2 ** 28, 2 ** 28, (M, N)).astype(np.int64)
    sw = (rng.random(N) * 1e-6).astype(np.float32)
    bf = rng.standard_normal(N).astype(np.float32)
    zn = rng.standard_normal(N).astype(np.float32)
    rn = (rng.random(N) * 50 + 1).astype(np.float32)
    q = oracle.epilogue_quantize(acc, sw, bf, zn, rn, 8, relu)
    for m in range(M):
        for n in range(N):
            a = frac_to_f32(Fraction(int(acc[m, n])))
            v = frac_to_f32(a * Fraction(float(sw[n])) + Fraction(float(bf[n])))
            if relu and not v > 0:
                v = Fraction(0)
            t = frac_to_f32(v - Fraction(float(zn[n])))
            u = frac_to_f32(t * Fraction(float(rn[n])))
            assert q[m, n] == max(-127, min(127, round(u)))


def test_epilogue_quantize_dyadic_exact():
    """Power-of-two scales and integer offsets: codes are exact rationals."""
    acc = np.array([[40, -40, 7, 1000, -3]], np.int64)
    sw = np.full(5, 0.25, np.float32)
    bf = np.array([1, 2, -0.5, 0, 3], np.float32)
    zn = np.array([0.5, -1, 0, 2, 0], np.float32)
    rn = np.array([2, 4, 8, 1, 16], np.float32)
    q = oracle.epilogue_quantize(acc, sw, bf, zn, rn, 8, relu=True)
    want = []
    for n in range(5):
        v = max(Fraction(int(acc[0, n])) * Fraction(1, 4) + Fraction(float(bf[n])), Fraction(0))
        want.append(max(-127, min(127, round((v - Fraction(float(zn[n]))) * Fraction(float(rn[n]))))))
    assert list(q[0]) == want


def test_epilogue_quantize_matches_unfused_chain_away_from_ties():
    """Fused codes = quantize(fp16 y) of the unfused chain, except where the
    fp16 rounding of y moves the value across a rounding boundary."""
    rng = np.random.default_rng(5)
    M, N = 64, 512
    acc = rng.integers(-2 ** 20, 2 ** 20, (M, N)).astype(np.int64)
    sw = (rng.random(N) * 2e-5).astype(np.float32)
    bf = (rng.standard_normal(N) * 0.5).astype(np.float32)
    y = oracle.epilogue(acc, sw, bf, relu=True)                 # fp16
    mn, mx = oracle.calibrate(y)
    zn, _, rn = oracle.params(mn, mx, 8)
    fused = oracle.epilogue_quantize(acc, sw, bf, zn, rn, 8, relu=True)
    unfused = oracle.quantize(y, zn, rn, 8)
    v = np.maximum(acc * sw.astype(np.float64) + bf.astype(np.float64), 0)
    u = (v - zn.astype(np.float64)) * rn.astype(np.float64)
    # fp16 rounding of y moves u by at most half an fp16 ulp of y times r
    ulp = np.spacing(np.abs(y).astype(np.float16)).astype(np.float64)
    slack = ulp * rn.astype(np.float64) / 2 + 1e-4
    far = np.abs(np.abs(u - np.floor(u)) - 0.5) > slack
    assert np.array_equal(fused[far], unfused[far])
    assert np.all(np.abs(fused.astype(np.int64) - unfused.astype(np.int64)) <= 1)
    assert far.mean() > 0.9
