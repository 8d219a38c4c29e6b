"""Pins of the oracle's token-wise clipping calibration (Appendix D: the static
activation scales of bias-free models are calibrated with token-wise clipping
after Outlier Suppression; reading: per-channel order statistics over the
calibration tokens at quantile alpha)."""
import numpy as np
import pytest

import oracle


def _np_clip(x, alpha):
    """numpy's inverted-CDF quantile (the smallest value whose empirical CDF
    reaches alpha) for the upper end, and of the negated data for the lower."""
    xf = x.astype(np.float64)
    hi = [np.quantile(c[~np.isnan(c)], alpha, method="inverted_cdf") for c in xf.T]
    lo = [-np.quantile(-c[~np.isnan(c)], alpha, method="inverted_cdf") for c in xf.T]
    return np.array(lo, np.float32), np.array(hi, np.float32)


@pytest.mark.parametrize("T,alpha", [(1000, 0.99), (4096, 0.999), (777, 0.9), (65, 0.5), (3, 0.999), (1, 0.99)])
def test_clipped_range_is_the_library_quantile(T, alpha):
    rng = np.random.default_rng(T)
    K = 24
    x = rng.standard_normal((T, K)) * np.exp(rng.standard_normal(K))
    x[rng.random((T, K)) < 0.01] *= 50                     # token outliers
    x = x.astype(np.float16)
    lo, hi = oracle.calibrate_clipped(x, alpha)
    lo_n, hi_n = _np_clip(x, alpha)
    assert np.array_equal(lo, lo_n) and np.array_equal(hi, hi_n)


def test_alpha_one_is_min_max_calibration():
    rng = np.random.default_rng(2)
    x = (rng.standard_normal((513, 40)) * 7).astype(np.float16)
    lo, hi = oracle.calibrate_clipped(x, 1.0)
    mn, mx = oracle.calibrate(x)
    assert np.array_equal(lo, mn) and np.array_equal(hi, mx)


def test_clipping_brute_force_and_nan():
    """Order statistics by brute-force counting, NaN ignored, signed zeros."""
    x = np.array([[3, -1, np.nan],
                  [1, -0.0, np.nan],
                  [2, 0.0, np.nan],
                  [-5, 7, np.nan],
                  [4, -0.0, 2]], np.float16)
    lo, hi = oracle.calibrate_clipped(x, 0.8)
    # column 0: sorted -5 1 2 3 4, T' = 5, rho = 4: hi = 3, lo = rank 2 = 1
    assert (lo[0], hi[0]) == (1, 3)
    # column 1: -1 -0 -0 0 7: rho = 4 -> hi = +0 (rank 4), lo = rank 2 = -0
    assert hi[1] == 0 and not np.signbit(hi[1]) and lo[1] == 0 and np.signbit(lo[1])
    # column 2: one non-NaN value
    assert (lo[2], hi[2]) == (2, 2)
    lo, hi = oracle.calibrate_clipped(x[:4, 2:], 0.9)        # only NaN: empty channel
    assert np.isposinf(lo[0]) and np.isneginf(hi[0])


def test_clipping_cuts_the_token_outliers_from_the_scale():
    """Clipping a few outlier tokens shrinks the channel scales and lowers the
    quantization error of the ordinary tokens (the reason Appendix D clips)."""
    rng = np.random.default_rng(9)
    T, K = 4096, 64
    x = rng.standard_normal((T, K))
    x[rng.choice(T, 4, replace=False)] *= 60                  # 4 outlier tokens
    x = x.astype(np.float16)
    mn, mx = oracle.calibrate(x)
    lo, hi = oracle.calibrate_clipped(x, 0.999)
    _, s_mm, r_mm = oracle.params(mn, mx, 6, symmetrize=False)
    _, s_cl, r_cl = oracle.params(lo, hi, 6, symmetrize=False)
    assert np.all(s_cl < s_mm)
    z0 = np.zeros(K, np.float32)
    ordinary = x[np.all(np.abs(x.astype(np.float64)) < 8, axis=1)]
    err = lambda s, r: np.abs(oracle.quantize(ordinary, z0, r, 6) * s.astype(np.float64) -
                              ordinary.astype(np.float64)).mean()
    assert err(s_cl, r_cl) < 0.5 * err(s_mm, r_mm)
