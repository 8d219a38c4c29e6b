"""Pins of the oracle's asymmetric per-output-channel weights (the paper's "Int8":
zero points for the weights, min-max calibration; Eq. 1 with z != 0)."""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from test_oracle_pins import frac_to_f32, frac_to_half


@pytest.mark.parametrize("bits", [8, 6, 4])
def test_asym_codes_dyadic_exact(bits):
    """Rows on a power-of-two grid lo + j * step, j = 0 .. 2^b - 1 in shuffled
    order: every fp32 step is exact, so the codes are j, the zero point is
    -lo / step, and (u - zp) * sw reproduces each weight exactly."""
    umax = (1 << bits) - 1
    shift = 1 << (bits - 1)
    rng = np.random.default_rng(bits)
    rows, zps = [], []
    for zp in (0, 1, umax // 3, umax - 1, umax):
        step = 2.0 ** -6
        vals = (np.arange(umax + 1) - zp) * step
        rng.shuffle(vals)
        rows.append(vals)
        zps.append(zp)
    w = np.array(rows, np.float16)
    assert np.all(w.astype(np.float64) == np.array(rows))  # exact in fp16
    qw, sw, zc = oracle.fold_codes_asym(w, None, bits)
    for i, zp in enumerate(zps):
        assert sw[i] == np.float32(2.0 ** -6)
        assert zc[i] == zp - shift
        u = qw[i].astype(np.int64) + shift
        assert np.array_equal(u, np.round(w[i].astype(np.float64) / 2.0 ** -6).astype(np.int64) + zp)
        assert np.all((u - zp) * 2.0 ** -6 == w[i].astype(np.float64))


def test_asym_codes_with_channel_scales_dyadic():
    """W_s = W (.) s with power-of-two s: the fold's product is exact, so the
    codes of W with scales s equal the codes of the pre-multiplied weights."""
    rng = np.random.default_rng(3)
    w = (rng.integers(-40, 90, (6, 32)) * 2.0 ** -5).astype(np.float16)
    s = (2.0 ** rng.integers(-3, 3, 32)).astype(np.float32)
    qa, swa, zca = oracle.fold_codes_asym(w, s, 8)
    ws = (w.astype(np.float64) * s).astype(np.float16)
    assert np.all(ws.astype(np.float64) == w.astype(np.float64) * s)
    qb, swb, zcb = oracle.fold_codes_asym(ws, None, 8)
    assert np.array_equal(qa, qb) and np.array_equal(swa, swb) and np.array_equal(zca, zcb)


@pytest.mark.parametrize("bits", [8, 6])
def test_asym_error_bound_range_and_zero(bits):
    umax = (1 << bits) - 1
    shift = 1 << (bits - 1)
    rng = np.random.default_rng(10 + bits)
    N, K = 40, 257
    w = rng.standard_normal((N, K)) * 0.02
    w[: N // 2] += rng.random((N // 2, 1)) * 0.05          # skewed rows
    w[:, 7] = 0.0                                         # an exact zero in every row
    w = w.astype(np.float16)
    qw, sw, zc = oracle.fold_codes_asym(w, None, bits)
    wf = w.astype(np.float64)
    u = qw.astype(np.int64) + shift
    zp = zc.astype(np.int64) + shift
    assert u.min() >= 0 and u.max() <= umax
    assert np.all((zp >= 0) & (zp <= umax))
    deq = (u - zp[:, None]) * sw.astype(np.float64)[:, None]
    # half a step, with room for the fp32 roundings of w * rw
    assert np.all(np.abs(deq - wf) <= sw.astype(np.float64)[:, None] * (0.5 + 1e-5))
    assert np.all(u[:, 7] == zp)                          # zero is represented exactly
    lo = np.minimum(wf.min(1), 0.0)
    hi = np.maximum(wf.max(1), 0.0)
    assert np.allclose(sw, (hi - lo) / umax, rtol=2 ** -22)
    for n in range(N):
        if wf[n].min() < 0:
            assert u[n, np.argmin(wf[n])] == 0                # round(lo r) = -round(-lo r)
        assert u[n, np.argmax(wf[n])] >= umax - 1


def test_asym_degenerate_rows():
    w = np.zeros((3, 16), np.float16)
    w[1] = np.linspace(0.1, 0.9, 16).astype(np.float16)   # all positive: zero point 0
    w[2] = -np.linspace(0.1, 0.9, 16).astype(np.float16)  # all negative: zero point 2^b - 1
    qw, sw, zc = oracle.fold_codes_asym(w, None, 8)
    assert sw[0] == 0 and np.all(qw[0] == zc[0])          # all-zero row: every code its zero point
    assert zc[1] == -128 and qw[1].max() == 127
    assert zc[2] == 127 and qw[2].min() == -128


def test_asym_product_identity_brute_force():
    """sum_k q (qw - zc) == acc - zc * rowsum, element by element in Python."""
    rng = np.random.default_rng(5)
    M, N, K = 3, 4, 37
    q = rng.integers(-127, 128, (M, K)).astype(np.int8)
    w = (rng.standard_normal((N, K)) * 0.05 + 0.02).astype(np.float16)
    qw, sw, zc = oracle.fold_codes_asym(w, None, 8)
    acc = oracle.matmul(q, qw)
    rs = oracle.rowsum(q)
    for m in range(M):
        assert rs[m] == sum(int(v) for v in q[m])
        for n in range(N):
            direct = sum(int(q[m, k]) * (int(qw[n, k]) - int(zc[n])) for k in range(K))
            assert direct == acc[m, n] - int(zc[n]) * rs[m]


def test_asym_epilogue_exact_rounding():
    rng = np.random.default_rng(29)
    M, N = 5, 7
    acc = rng.integers(-2 ** 30, 2 ** 30, (M, N)).astype(np.int64)
    rs = rng.integers(-2 ** 20, 2 ** 20, M).astype(np.int64)
    zc = rng.integers(-128, 128, N).astype(np.int32)
    sw = (rng.random(N) * 1e-4).astype(np.float32)
    b = rng.standard_normal(N).astype(np.float32)
    for relu in (False, True):
        y = oracle.epilogue_asym(acc, rs, zc, sw, b, relu).astype(np.float64)
        for m in range(M):
            for n in range(N):
                t = int(acc[m, n]) - int(zc[n]) * int(rs[m])          # exact integer
                a = frac_to_f32(Fraction(t))
                v = frac_to_f32(a * Fraction(float(sw[n])) + Fraction(float(b[n])))
                if relu and not v > 0:
                    v = Fraction(0)
                e = frac_to_half(v)
                assert y[m, n] == e or (math.isinf(e) and y[m, n] == e)


def test_asym_beats_symmetric_on_one_sided_rows():
    """The "Int8" weights trade speed for accuracy (Section 4): on rows whose
    values are one-sided the zero point uses the whole code range, so the
    reconstruction error of W_s falls well below the symmetric codes'."""
    rng = np.random.default_rng(41)
    N, K = 64, 512
    w = (rng.random((N, K)) * 0.04 + 0.01).astype(np.float16)   # all in [0.01, 0.05]
    z = np.zeros(K, np.float32)
    s = np.ones(K, np.float32)
    for bits in (8, 6):
        qs, sws, _ = oracle.fold(w, None, z, s, bits)
        qa, swa, zca = oracle.fold_codes_asym(w, None, bits)
        wf = w.astype(np.float64)
        err_sym = np.abs(qs * sws.astype(np.float64)[:, None] - wf).mean()
        err_asym = np.abs((qa.astype(np.int64) - zca[:, None]) * swa.astype(np.float64)[:, None] - wf).mean()
        assert err_asym < 0.6 * err_sym
