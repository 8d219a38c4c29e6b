"""GPU parity at the workloads' full sizes (the launch configurations the
benchmark times): the CUDA path runs the whole layer; the oracle checks a
sample of rows and output channels (codes, int32 accumulators, fp16 outputs)
plus the per-channel parameters and folded weights of the sampled channels."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_f16_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


CASES = [
    # (config, layer index, tokens, calibration tokens)
    (1, 0, 16, 64),
    (2, 0, 2048, 65536), (2, 1, 2048, 8192), (2, 2, 2048, 8192), (2, 3, 2048, 8192),
    (3, 0, 1, 4096), (3, 0, 16, 4096), (3, 0, 128, 4096), (3, 0, 1024, 4096), (3, 0, 4096, 4096),
    (3, 1, 16, 4096), (3, 2, 1024, 4096), (3, 3, 1, 4096), (3, 3, 4096, 4096),
    (4, 0, 4096, 4096), (4, 1, 4096, 4096),
    (5, 0, 4096, 4096), (5, 1, 4096, 4096), (5, 2, 4096, 4096), (5, 3, 4096, 4096),
]


def _run(cfg, li, M, T, bits):
    from paper_2406_18832_gb300 import QuantizedLinear, binding, synth
    dev = torch.device("cuda")
    c = synth.CONFIGS[cfg]
    layer = c.layers[li]
    bits_a, bits_w = bits
    w, b = synth.weights(cfg, li, layer, device=dev)
    xc = synth.activations(cfg, li, layer, T, 3, device=dev)
    x = synth.activations(cfg, li, layer, M, 4, device=dev)
    ql = QuantizedLinear(layer.K, layer.N, bits_a, bits_w, relu=layer.relu_out, device=dev)
    ql.calibrate(xc).fold(w, b)
    q = ql.quantize(x)
    y = ql.linear(q)
    acc = torch.empty(M, layer.N, dtype=torch.int32, device=dev)
    binding.ot_linear_s32(q, ql.qw, bits_a, bits_w, acc)
    torch.cuda.synchronize()
    assert binding.ot_get_device_status() == binding.OT_OK

    rng = np.random.default_rng(cfg * 1000 + li * 10 + M)
    rows = np.unique(np.concatenate([[0, M - 1], rng.choice(M, min(M, 24), replace=False)]))
    cols = np.unique(np.concatenate([[0, layer.N - 1], rng.choice(layer.N, min(layer.N, 256), replace=False)]))
    rows_t = torch.from_numpy(rows).to(dev)
    cols_t = torch.from_numpy(cols).to(dev)

    mn, mx = oracle.calibrate(xc.cpu().numpy())
    z, s, r = oracle.params(mn, mx, bits_a)
    assert np.array_equal(ql.ch_min.cpu().numpy(), mn) and np.array_equal(ql.ch_max.cpu().numpy(), mx)
    assert np.array_equal(ql.z.cpu().numpy(), z) and np.array_equal(ql.s.cpu().numpy(), s)
    assert np.array_equal(ql.r.cpu().numpy(), r)
    wc = w.index_select(0, cols_t).cpu().numpy()
    bc = b.index_select(0, cols_t).cpu().numpy()
    qw, sw, bf = oracle.fold(wc, bc, z, s, bits_w)
    assert np.array_equal(ql.qw.index_select(0, cols_t).cpu().numpy(), qw)
    assert np.array_equal(ql.sw.index_select(0, cols_t).cpu().numpy(), sw)
    assert np.array_equal(ql.b_fold.index_select(0, cols_t).cpu().numpy(), bf)
    xr = x.index_select(0, rows_t).cpu().numpy()
    oq = oracle.quantize(xr, z, r, bits_a)
    assert np.array_equal(q.index_select(0, rows_t).cpu().numpy().astype(np.int64), oq.astype(np.int64))
    oacc = oracle.matmul(oq, qw)
    gacc = acc.index_select(0, rows_t).index_select(1, cols_t).cpu().numpy().astype(np.int64)
    assert np.array_equal(gacc, oacc)
    oy = oracle.epilogue(oacc, sw, bf, layer.relu_out)
    gy = y.index_select(0, rows_t).index_select(1, cols_t).cpu().numpy()
    assert_f16_close(gy, oy)
    # properties over the whole output: finite, and ReLU outputs non-negative
    assert torch.isfinite(y).all()
    if layer.relu_out:
        assert (y >= 0).all()


@pytest.mark.parametrize("cfg,li,M,T", CASES)
def test_full_size_layer(cfg, li, M, T):
    from paper_2406_18832_gb300 import synth
    bits = synth.CONFIGS[cfg].bits[0]
    _run(cfg, li, M, T, bits)


@pytest.mark.parametrize("li", [0, 2])
def test_config5_int6(li):
    _run(5, li, 4096, 4096, (6, 6))


def test_device_timeout_status_and_recovery():
    """A bounded device wait that nothing satisfies records OT_ERR_TIMEOUT,
    the status clears once read, and the context keeps working."""
    from paper_2406_18832_gb300 import binding
    assert binding.ot_get_device_status() == binding.OT_OK
    binding.ot_selftest_wait_timeout(50_000_000)
    assert binding.ot_get_device_status() == binding.OT_ERR_TIMEOUT
    assert binding.ot_get_device_status() == binding.OT_OK
    q = torch.ones(32, 64, dtype=torch.float16, device="cuda")
    qw = torch.ones(16, 64, dtype=torch.int8, device="cuda")
    acc = torch.empty(32, 16, dtype=torch.int32, device="cuda")
    binding.ot_linear_s32(q, qw, 8, 8, acc)
    torch.cuda.synchronize()
    assert torch.all(acc == 64)
    assert binding.ot_get_device_status() == binding.OT_OK
