"""Token-wise clipping calibration (Appendix D) on the GPU against the oracle:
per-channel order statistics, bit for bit, then a bias-free layer calibrated
with it end to end."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _tokens(T, K, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, K)) * np.exp(rng.standard_normal(K))
    x[rng.random((T, K)) < 0.002] *= 80                       # outlier tokens
    return x.astype(np.float16)


@pytest.mark.parametrize("T,K,pad", [(1, 1, 0), (3, 33, 0), (1000, 64, 8), (8192, 4096, 0), (70000, 40, 0)])
@pytest.mark.parametrize("alpha", [1.0, 0.999, 0.9, 0.5])
def test_calibrate_clipped_bit_exact(T, K, pad, alpha):
    from paper_2406_18832_gb300 import binding as B
    x = _tokens(T, K, T + K)
    if T >= 3:
        x[1, :] = -0.0
        x[2, : K // 2] = np.nan
    lo_o, hi_o = oracle.calibrate_clipped(x, alpha)
    xb = torch.zeros(T, K + pad, dtype=torch.float16)
    xb[:, :K] = torch.as_tensor(x)
    lo = torch.full((K,), 7.0, device=DEV)
    hi = torch.full((K,), 7.0, device=DEV)
    B.ot_calibrate_clipped(xb.to(DEV)[:, :K], alpha, lo, hi)
    assert np.array_equal(lo.cpu().numpy().view(np.uint32), lo_o.view(np.uint32))
    assert np.array_equal(hi.cpu().numpy().view(np.uint32), hi_o.view(np.uint32))


def test_calibrate_clipped_all_nan_channel():
    from paper_2406_18832_gb300 import binding as B
    x = np.full((50, 3), np.nan, np.float16)
    x[:, 1] = np.arange(50)
    lo = torch.empty(3, device=DEV)
    hi = torch.empty(3, device=DEV)
    B.ot_calibrate_clipped(torch.as_tensor(x).to(DEV), 0.9, lo, hi)
    lo, hi = lo.cpu().numpy(), hi.cpu().numpy()
    assert np.isposinf(lo[0]) and np.isneginf(hi[0]) and (lo[1], hi[1]) == (5, 44)


def test_bias_free_layer_with_clipping_end_to_end():
    """QuantizedLinear(symmetrize=False).calibrate_clipped -> fold -> forward
    equals the oracle chain (clipped range, z = 0 params, fold, quantize,
    product, epilogue)."""
    from paper_2406_18832_gb300 import QuantizedLinear
    T, M, N, K = 4096, 48, 256, 512
    x_cal, x = _tokens(T, K, 1), _tokens(M, K, 2)
    rng = np.random.default_rng(3)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float16)
    ql = QuantizedLinear(K, N, 6, 6, symmetrize=False, device=DEV)
    ql.calibrate_clipped(torch.as_tensor(x_cal).to(DEV), 0.999).fold(torch.as_tensor(w).to(DEV), None)
    y = ql(torch.as_tensor(x).to(DEV)).cpu().numpy()
    lo, hi = oracle.calibrate_clipped(x_cal, 0.999)
    z, s, r = oracle.params(lo, hi, 6, symmetrize=False)
    assert np.all(z == 0)
    qw, sw, bf = oracle.fold(w, None, z, s, 6)
    ref = oracle.epilogue(oracle.matmul(oracle.quantize(x, z, r, 6), qw), sw, bf)
    assert np.array_equal(y.view(np.uint16), ref.view(np.uint16))
