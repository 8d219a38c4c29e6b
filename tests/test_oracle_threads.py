"""The oracle's threaded drivers (used for full-size parity and the CPU
baseline) return exactly what its single-threaded functions return."""
import numpy as np

import oracle


def test_threaded_drivers_equal_single_threaded():
    rng = np.random.default_rng(11)
    x = (rng.standard_normal((301, 520)) * 7).astype(np.float16)
    x[5, 7] = np.nan
    mn, mx = oracle.calibrate(x)
    for a, b in zip(oracle.calibrate_mt(x, threads=5), (mn, mx)):
        assert np.array_equal(a, b, equal_nan=True)
    # running calibration continues from given min / max
    m0 = oracle.calibrate(x[:100])
    for a, b in zip(oracle.calibrate_mt(x[100:], *m0, threads=3), oracle.calibrate(x[100:], *m0)):
        assert np.array_equal(a, b)
    z, s, r = oracle.params(mn, mx, 8)
    w = (rng.standard_normal((131, 520)) * 0.02).astype(np.float16)
    b = (rng.standard_normal(131) * 0.01).astype(np.float16)
    for a, c in zip(oracle.fold_mt(w, b, z, s, 6, threads=4), oracle.fold(w, b, z, s, 6)):
        assert np.array_equal(a, c)
    q = oracle.quantize(x, z, r, 8)
    assert np.array_equal(oracle.quantize_mt(x, z, r, 8, threads=7), q)
    qw, sw, bf = oracle.fold(w, b, z, s, 8)
    acc = oracle.matmul(q, qw)
    assert np.array_equal(oracle.matmul_mt(q, qw, threads=6), acc)        # split over tokens
    assert np.array_equal(oracle.matmul_mt(q[:2], qw, threads=6), acc[:2])  # split over channels
    assert np.array_equal(oracle.epilogue_mt(acc, sw, bf, True, threads=4).view(np.uint16),
                          oracle.epilogue(acc, sw, bf, True).view(np.uint16))
