"""Pins of the oracle's LayerNorm fused with the symmetrization and the
per-channel quantization (Section 3.2: the codes round((LN(h) - z) / s) come
out of the LayerNorm kernel, with LN's gamma and beta absorbing r and z)."""
from fractions import Fraction

import numpy as np
import pytest

import oracle


def _ln_ref(h, gamma, beta, eps):
    """LayerNorm in fp64 with numpy (biased variance)."""
    x = h.astype(np.float64)
    mu = x.mean(axis=1, keepdims=True)
    var = x.var(axis=1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * gamma.astype(np.float64) + beta.astype(np.float64), mu[:, 0], var[:, 0]


def test_ln_statistics_match_fp64_library():
    """mean and 1/sqrt(var + eps) from the exact integer sums agree with numpy's
    fp64 mean / variance to within the fp32 roundings of their definition
    (mean: 2 roundings; rstd: at most 7 from the exact variance), over rows
    with large, small, subnormal and mixed-sign values."""
    rng = np.random.default_rng(1)
    K = 1536
    rows = [rng.standard_normal(K), rng.standard_normal(K) * 1000 + 3000, rng.standard_normal(K) * 1e-3,
            rng.standard_normal(K) * 6e-8, np.concatenate([np.full(K - 8, 0.5), rng.standard_normal(8) * 60]),
            np.linspace(-65000, 65000, K)]
    h = np.array(rows).astype(np.float16)
    gr, br = oracle.fold_layernorm(np.ones(K, np.float16), np.zeros(K, np.float16), np.zeros(K, np.float32),
                                   np.ones(K, np.float32))
    eps = 1e-5
    _, mean, rstd = oracle.layernorm_quantize(h, gr, br, eps, 8)[1:]
    _, mu, var = _ln_ref(h, np.ones(K), np.zeros(K), eps)
    assert np.all(np.abs(mean.astype(np.float64) - mu) <= np.abs(mu) * 2 * 2 ** -24 * 1.0001)
    want = 1 / np.sqrt(var + np.float64(np.float32(eps)))
    assert np.all(np.abs(rstd.astype(np.float64) - want) <= want * 7 * 2 ** -24)


@pytest.mark.parametrize("a,c,eps", [(1.5, 0.25, 1.75), (4.0, -2.0, 0.0), (0.125, 64.0, 0.046875)])
def test_ln_fused_codes_dyadic_exact(a, c, eps):
    """Rows c +- a (alternating): mean c and biased variance a^2 exactly, and
    var + eps a power-of-two square, so every step is exact and the codes are
    round(+-gamma r / sqrt(a^2 + eps) + (beta - z) r) as rationals.  Adding eps
    outside the square root, or the unbiased variance, would change them."""
    K = 64
    h = np.array([[c + a if k % 2 == 0 else c - a for k in range(K)]], np.float16)
    assert h.astype(np.float64).mean() == c and h.astype(np.float64).var() == a * a
    s2 = Fraction(a) ** 2 + Fraction(eps)
    root = Fraction(int(s2.numerator ** 0.5), int(s2.denominator ** 0.5))
    assert root * root == s2                                  # the case is exact
    rng = np.random.default_rng(7)
    gamma = (2.0 ** rng.integers(-2, 3, K) * rng.choice([-1, 1], K)).astype(np.float16)
    beta = (rng.integers(-8, 9, K) * 0.25).astype(np.float16)
    z = (rng.integers(-8, 9, K) * 0.125).astype(np.float32)
    r = (2.0 ** rng.integers(0, 4, K)).astype(np.float32)
    gr, br = oracle.fold_layernorm(gamma, beta, z, r)
    q, rs, mean, rstd_o = oracle.layernorm_quantize(h, gr, br, np.float32(eps), 8)
    assert Fraction(float(mean[0])) == Fraction(c) and Fraction(float(rstd_o[0])) == 1 / root
    for k in range(K):
        n = (Fraction(float(h[0, k])) - Fraction(c)) / root
        u = n * Fraction(float(gamma[k])) * Fraction(float(r[k])) + \
            (Fraction(float(beta[k])) - Fraction(float(z[k]))) * Fraction(float(r[k]))
        assert q[0, k] == max(-127, min(127, round(u)))       # round half to even
    assert rs[0] == int(q[0].astype(np.int64).sum())


def test_ln_statistics_every_fp16_value_exact_rational():
    """Every fp16 bit pattern: one row per exponent field (all 2048 patterns of
    that exponent, both signs), then every finite value once over rows of
    4096.  The exact mean and biased variance of each row, in rationals from
    the fp16 values themselves, bound the oracle's fp32 mean (2 roundings) and
    1/sqrt(var + eps) (at most 7), from subnormals to 65504."""
    rng = np.random.default_rng(5)
    pats = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    exp = (pats >> 10) & 31
    rows = [rng.permutation(pats[exp == e]) for e in range(31)]
    fin = rng.permutation(pats[exp != 31])
    allv = np.zeros(-(-fin.size // 4096) * 4096, np.uint16)
    allv[: fin.size] = fin
    h_bands = np.stack(rows).view(np.float16)
    h_all = allv.reshape(-1, 4096).view(np.float16)
    eps = np.float32(1e-5)
    for h in (h_bands, h_all):
        K = h.shape[1]
        gr, br = oracle.fold_layernorm(np.ones(K, np.float16), np.zeros(K, np.float16), np.zeros(K, np.float32),
                                       np.ones(K, np.float32))
        _, _, mean, rstd = oracle.layernorm_quantize(h, gr, br, float(eps), 8)
        for i in range(h.shape[0]):
            vals = [Fraction(float(v)) for v in h[i].astype(np.float64)]
            mu = sum(vals) / K
            var = sum((v - mu) ** 2 for v in vals) / K
            assert abs(Fraction(float(mean[i])) - mu) <= abs(mu) * Fraction(2, 2 ** 24) * Fraction(10001, 10000)
            want = 1 / np.sqrt(float(var + Fraction(float(eps))))
            assert abs(float(rstd[i]) - want) <= want * 7 * 2 ** -24


def test_ln_fused_matches_unfused_away_from_ties():
    """The fused codes equal round((LN(h) - z) * r) computed in fp64 wherever
    the fp64 value is not within 1e-3 of a rounding boundary."""
    rng = np.random.default_rng(11)
    M, K = 48, 1024
    h = (rng.standard_normal((M, K)) * 2 + rng.standard_normal(K) * 0.5).astype(np.float16)
    h[:, :10] *= 30                                            # outlier channels
    gamma = (1 + 0.2 * rng.standard_normal(K)).astype(np.float16)
    beta = (0.1 * rng.standard_normal(K)).astype(np.float16)
    y, _, _ = _ln_ref(h, gamma, beta, 1e-5)
    mn, mx = oracle.calibrate(y.astype(np.float16))
    z, s, r = oracle.params(mn, mx, 8)
    gr, br = oracle.fold_layernorm(gamma, beta, z, r)
    q = oracle.layernorm_quantize(h, gr, br, 1e-5, 8)[0]
    u = (y - z.astype(np.float64)) * r.astype(np.float64)
    ref = np.clip(np.rint(u), -127, 127)
    far = np.abs(np.abs(u - np.floor(u)) - 0.5) > 1e-3
    assert np.array_equal(q[far], ref[far].astype(np.int8))
    assert np.all(np.abs(q.astype(np.int64) - ref) <= 1)
    assert far.mean() > 0.99


def test_ln_with_unit_affine_reduces_to_plain_quantizer():
    """gamma = 1, beta = z: the codes are round(n * r) of the normalized row."""
    rng = np.random.default_rng(3)
    M, K = 8, 512
    h = (rng.standard_normal((M, K)) * 3).astype(np.float16)
    z = (rng.standard_normal(K) * 0.5).astype(np.float16)
    r = np.full(K, 20.0, np.float32)
    gr, br = oracle.fold_layernorm(np.ones(K, np.float16), z, z.astype(np.float32), r)
    assert np.all(br == 0) and np.all(gr == 20)
    q, _, mean, rstd = oracle.layernorm_quantize(h, gr, br, 1e-5, 8)
    n = (h.astype(np.float32) - mean[:, None]) * rstd[:, None]           # fp32, as defined
    assert np.array_equal(q, np.clip(np.rint((n * np.float32(20)).astype(np.float32)), -127, 127).astype(np.int8))


def test_ln_nonfinite_row_codes_zero():
    K = 32
    h = np.ones((3, K), np.float16)
    h[0, 5] = np.inf
    h[1, 7] = np.nan
    h[2] = np.linspace(-1, 1, K).astype(np.float16)
    gr, br = oracle.fold_layernorm(np.ones(K, np.float16), np.zeros(K, np.float16), np.zeros(K, np.float32),
                                   np.full(K, 50, np.float32))
    q, rs, _, _ = oracle.layernorm_quantize(h, gr, br, 1e-5, 8)
    assert np.all(q[:2] == 0) and rs[0] == 0 and rs[1] == 0
    assert np.any(q[2] != 0)
