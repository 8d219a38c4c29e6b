"""Pins of the oracle's per-token path (Eq. 3; the paper's out / fc2 linears)."""
import math
from fractions import Fraction

import numpy as np

import oracle
from test_oracle_pins import frac_to_f32, frac_to_half


def test_per_token_codes_dyadic_exact():
    # rows whose max |x| is 127 (r = 1) or 63.5 (r = 2): every fp32 step is exact
    x = np.array([[127, -3.5, 2.5, 0.5, -126.5],
                  [63.5, 1.25, -0.75, 0.25, -63.5]], np.float16)
    q, s = oracle.quantize_tokens(x, 8)
    assert s[0] == np.float32(1) and s[1] == np.float32(0.5)
    for m, r in ((0, 1), (1, 2)):
        for k in range(5):
            assert q[m, k] == round(Fraction(float(x[m, k])) * r)  # half to even
    assert list(q[0]) == [127, -4, 2, 0, -126]


def test_per_token_invariants():
    rng = np.random.default_rng(21)
    x = (rng.standard_normal((40, 300)) * rng.uniform(0.01, 50, (40, 1))).astype(np.float16)
    x[3] = 0
    x[5, 7] = np.float16(np.nan)
    for bits in (8, 6, 4):
        qm = oracle.qmax(bits)
        q, s = oracle.quantize_tokens(x, bits)
        xf = x.astype(np.float64)
        amax = np.nanmax(np.abs(xf), axis=1)
        assert s[3] == 0 and np.all(q[3] == 0)
        assert q[5, 7] == 0
        live = amax > 0
        assert np.array_equal(s[live], (amax[live].astype(np.float32) / np.float32(qm)))
        assert np.all(np.abs(q[live]).max(1) == qm)      # the largest element reaches qmax
        r = np.where(live, np.float32(qm) / amax.astype(np.float32), 0).astype(np.float64)
        v = np.nan_to_num(xf) * r[:, None]
        assert np.all(np.abs(q - v) <= 0.5 + np.abs(v) * 2.0 ** -22)


def test_per_token_path_is_eq3():
    """Y = s^X_i s^W_j sum_k X~_ik W~_kj + b (Eq. 3), written independently in numpy."""
    rng = np.random.default_rng(22)
    M, K, N = 9, 256, 33
    x = (rng.standard_normal((M, K)) * 3).astype(np.float16)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float16)
    b = (rng.standard_normal(N) * 0.1).astype(np.float32)
    q, s = oracle.quantize_tokens(x, 8)
    qw, sw = oracle.quantize_weights(w, 8)
    # W~: per-output-channel symmetric codes of W itself (no activation scale)
    amax_w = np.abs(w.astype(np.float32)).max(1)
    assert np.array_equal(sw, amax_w / np.float32(127))
    wt = np.clip(np.rint(w.astype(np.float32) * (np.float32(127) / amax_w)[:, None]), -127, 127)
    assert np.array_equal(qw.astype(np.float32), wt)
    acc = oracle.matmul(q, qw)
    y = oracle.epilogue_tokens(acc, s, sw, b).astype(np.float64)
    y3 = s.astype(np.float64)[:, None] * sw.astype(np.float64)[None, :] * (q.astype(np.float64) @ qw.astype(np.float64).T) + b
    assert np.allclose(y, y3, rtol=2 ** -10, atol=2 ** -14)
    # and it approximates XW^T + b within the quantization error bound
    ref = x.astype(np.float64) @ w.astype(np.float64).T + b
    bound = (s.astype(np.float64)[:, None] * sw.astype(np.float64)[None, :]) * \
        (np.abs(q).sum(1)[:, None] / 2 + np.abs(qw).sum(1)[None, :] / 2 + K / 4)
    assert np.all(np.abs(y - ref) <= bound + np.abs(ref) * 2 ** -10 + 1e-3)


def test_per_token_epilogue_exact_rounding():
    rng = np.random.default_rng(23)
    acc = rng.integers(-2 ** 30, 2 ** 30, (5, 7)).astype(np.int64)
    s = (rng.random(5) * 1e-2).astype(np.float32)
    sw = (rng.random(7) * 1e-3).astype(np.float32)
    b = (rng.standard_normal(7)).astype(np.float32)
    y = oracle.epilogue_tokens(acc, s, sw, b).astype(np.float64)
    for m in range(5):
        for n in range(7):
            a = frac_to_f32(Fraction(int(acc[m, n])))
            sc = frac_to_f32(Fraction(float(s[m])) * Fraction(float(sw[n])))
            v = frac_to_f32(a * sc + Fraction(float(b[n])))
            e = frac_to_half(v)
            assert y[m, n] == e or (math.isinf(e) and y[m, n] == e)
