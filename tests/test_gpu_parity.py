"""GPU parity: every C-ABI entry point against the CPU oracle on seeded inputs.

Integer results (codes, int32 accumulators) and the fp32 parameters (min,
max, z, s, r, sw, b') are compared bit for bit; fp16 outputs within
max(1 fp16 ulp, 1e-3 * max|y|).  Shapes span several tiles with ragged
tails in every dimension.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_f16_close, compare_layer, gpu_layer, oracle_layer

pytestmark = pytest.mark.gpu

B = None


@pytest.fixture(scope="module", autouse=True)
def _lib():
    global B
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2406_18832_gb300 import binding
    B = binding
    yield


DEV = "cuda"


def _gen(seed):
    return torch.Generator().manual_seed(seed)


def _acts(T, K, seed, outliers=True):
    g = _gen(seed)
    x = torch.randn(T, K, generator=g)
    if outliers and K >= 8:
        idx = torch.randperm(K, generator=g)[: max(1, K // 100)]
        x[:, idx] = x[:, idx] * (20 + 60 * torch.rand(idx.numel(), generator=g)) + \
            (-20 + 40 * torch.rand(idx.numel(), generator=g))
    return x.half()


# --------------------------------------------------------------------------
# calibration and parameters
# --------------------------------------------------------------------------
@pytest.mark.parametrize("T,K", [(1, 8), (37, 768), (1000, 4104), (5000, 264)])
def test_calibrate_bit_exact(T, K):
    x = _acts(T, K, 11)
    mn = torch.empty(K, device=DEV)
    mx = torch.empty(K, device=DEV)
    B.ot_calibrate(x.to(DEV), mn, mx, reset=True)
    omn, omx = oracle.calibrate(x.numpy())
    assert np.array_equal(mn.cpu().numpy(), omn) and np.array_equal(mx.cpu().numpy(), omx)
    # streaming in two batches, the second through a strided view (ldx > K)
    big = torch.zeros(T, K + 24, dtype=torch.float16)
    big[:, :K] = x
    bd = big.to(DEV)
    h = T // 2
    B.ot_calibrate(bd[:h, :K], mn, mx, reset=True)
    B.ot_calibrate(bd[h:, :K], mn, mx, reset=False)
    assert np.array_equal(mn.cpu().numpy(), omn) and np.array_equal(mx.cpu().numpy(), omx)


def test_calibrate_ignores_nan_and_empty_batch():
    x = _acts(64, 16, 12)
    x[3, 5] = float("nan")
    x[7, 2] = float("inf")
    mn = torch.empty(16, device=DEV)
    mx = torch.empty(16, device=DEV)
    B.ot_calibrate(x.to(DEV), mn, mx, reset=True)
    B.ot_calibrate(x[:0].to(DEV), mn, mx, reset=False)
    omn, omx = oracle.calibrate(x.numpy())
    assert np.array_equal(mn.cpu().numpy(), omn) and np.array_equal(mx.cpu().numpy(), omx)


@pytest.mark.parametrize("bits", [8, 6, 4, 2])
@pytest.mark.parametrize("sym", [True, False])
def test_params_bit_exact(bits, sym):
    g = _gen(13)
    K = 1000
    lo = torch.randn(K, generator=g) * 30 - 10
    hi = lo + torch.rand(K, generator=g) * 50
    lo[:4] = torch.tensor([3.0, float("inf"), 0.0, -2.0])
    hi[:4] = torch.tensor([3.0, float("-inf"), 0.0, 6.0])
    z, s, r = (torch.empty(K, device=DEV) for _ in range(3))
    B.ot_derive_params(lo.to(DEV), hi.to(DEV), bits, z, s, r, symmetrize=sym)
    oz, os_, or_ = oracle.params(lo.numpy(), hi.numpy(), bits, sym)
    for a, b_ in ((z, oz), (s, os_), (r, or_)):
        assert np.array_equal(a.cpu().numpy(), b_)


# --------------------------------------------------------------------------
# fold
# --------------------------------------------------------------------------
@pytest.mark.parametrize("N,K,bits_w,bias", [(1, 16, 8, True), (17, 784, 8, False), (300, 4096, 6, True),
                                            (64, 36864, 8, True)])
def test_fold_bit_exact(N, K, bits_w, bias):
    g = _gen(14)
    W = (torch.randn(N, K, generator=g) * 0.02).half()
    W[0, : min(K, 5)] = 0
    b = (torch.randn(N, generator=g) * 0.01).half() if bias else None
    xc = _acts(256, K, 15)
    f32 = dict(device=DEV, dtype=torch.float32)
    mn, mx = torch.empty(K, **f32), torch.empty(K, **f32)
    B.ot_calibrate(xc.to(DEV), mn, mx)
    z, s, r = (torch.empty(K, **f32) for _ in range(3))
    qw = torch.empty(N, K, dtype=torch.int8, device=DEV)
    sw, bf = torch.empty(N, **f32), torch.empty(N, **f32)
    B.ot_fold_weights(mn, mx, 8, W.to(DEV), None if b is None else b.to(DEV), bits_w, z, s, r, qw, sw, bf)
    omn, omx = oracle.calibrate(xc.numpy())
    oz, os_, _ = oracle.params(omn, omx, 8)
    oqw, osw, obf = oracle.fold(W.numpy(), None if b is None else b.numpy(), oz, os_, bits_w)
    assert np.array_equal(qw.cpu().numpy(), oqw)
    assert np.array_equal(sw.cpu().numpy(), osw)
    assert np.array_equal(bf.cpu().numpy(), obf)


# --------------------------------------------------------------------------
# quantize
# --------------------------------------------------------------------------
@pytest.mark.parametrize("M,K,pad", [(1, 8, 0), (3, 768, 8), (64, 264, 0), (65, 4104, 16), (1000, 512, 0)])
@pytest.mark.parametrize("bits", [8, 6])
def test_quantize_bit_exact(M, K, pad, bits):
    x = _acts(M, K, 16)
    xc = _acts(200, K, 17)
    if M > 2:
        x[1, 0] = float("nan")
        x[2, 0] = float("inf")
        x[2, 1] = float("-inf")
    omn, omx = oracle.calibrate(xc.numpy())
    oz, os_, or_ = oracle.params(omn, omx, bits)
    xb = torch.zeros(M, K + pad, dtype=torch.float16)
    xb[:, :K] = x
    xd = xb.to(DEV)[:, :K]
    z, r = torch.from_numpy(oz).to(DEV), torch.from_numpy(or_).to(DEV)
    q16 = torch.empty(M, K, dtype=torch.float16, device=DEV)
    q8 = torch.empty(M, K, dtype=torch.int8, device=DEV)
    B.ot_quantize_act(xd, z, r, bits, q16, B.OT_CODE_F16)
    B.ot_quantize_act(xd, z, r, bits, q8, B.OT_CODE_I8)
    oq = oracle.quantize(x.numpy(), oz, or_, bits)
    assert np.array_equal(q8.cpu().numpy(), oq)
    q16n = q16.cpu().numpy()
    assert np.array_equal(q16n.astype(np.int64), oq.astype(np.int64))
    assert np.array_equal(q16n, oq.astype(np.float16))  # exact integers, +0 for code 0


# --------------------------------------------------------------------------
# the integer product and the epilogue
# --------------------------------------------------------------------------
def _codes(shape, qmax, seed):
    g = _gen(seed)
    return torch.randint(-qmax, qmax + 1, shape, generator=g, dtype=torch.int32)


SHAPES = [(1, 16, 16), (5, 128, 64), (16, 144, 80), (17, 256, 1040), (33, 130, 2048), (64, 384, 1024),
          (100, 272, 4096), (128, 128, 1088), (200, 500, 640), (300, 1024, 2112), (1030, 144, 256)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits", [(8, 8), (6, 6)])
def test_linear_s32_bit_exact(M, N, K, bits):
    ba, bw = bits
    qa, qwm = (1 << (ba - 1)) - 1, (1 << (bw - 1)) - 1
    q = _codes((M, K), qa, 21 + M)
    qw = _codes((N, K), qwm, 22 + N)
    acc = torch.empty(M, N, dtype=torch.int32, device=DEV)
    B.ot_linear_s32(q.half().to(DEV), qw.to(torch.int8).to(DEV), ba, bw, acc)
    ref = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    got = acc.cpu().numpy().astype(np.int64)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("K", [1024, 1088, 4096, 16384])
def test_linear_s32_adversarial_extremes(K):
    """All-+-127 rows: partial sums sit at the edge of fp32 exactness inside a
    chunk and the totals need the int32 carry across chunks."""
    M, N = 4, 256
    q = torch.full((M, K), 127, dtype=torch.int32)
    q[1] = -127
    q[2, ::2] = -127
    q[3] = torch.where(torch.arange(K) % 3 == 0, 127, -126)
    qw = torch.full((N, K), 127, dtype=torch.int32)
    qw[1::2] = -127
    qw[5, K // 2:] = 1
    acc = torch.empty(M, N, dtype=torch.int32, device=DEV)
    B.ot_linear_s32(q.half().to(DEV), qw.to(torch.int8).to(DEV), 8, 8, acc)
    ref = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)


@pytest.mark.parametrize("M,N,K", [(16, 768, 768), (100, 272, 4096), (300, 1000, 512)])
@pytest.mark.parametrize("relu", [False, True])
def test_linear_f16_within_tolerance(M, N, K, relu):
    q = _codes((M, K), 127, 31)
    qw = _codes((N, K), 127, 32)
    g = _gen(33)
    sw = (torch.rand(N, generator=g) * 1e-4).float()
    bf = (torch.randn(N, generator=g) * 2).float()
    ld = N + 8
    ybig = torch.full((M, ld), 7.0, dtype=torch.float16, device=DEV)
    y = ybig[:, :N]
    B.ot_linear(q.half().to(DEV), qw.to(torch.int8).to(DEV), sw.to(DEV), bf.to(DEV), 8, 8, y, relu=relu)
    acc = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    ref = oracle.epilogue(acc, sw.numpy(), bf.numpy(), relu)
    assert_f16_close(y.cpu().numpy(), ref)
    assert torch.all(ybig[:, N:] == 7.0)  # padding columns untouched


def test_zero_token_batch():
    qw = torch.zeros(16, 64, dtype=torch.int8, device=DEV)
    y = torch.empty(0, 16, dtype=torch.float16, device=DEV)
    q = torch.empty(0, 64, dtype=torch.float16, device=DEV)
    B.ot_linear(q, qw, torch.ones(16, device=DEV), torch.zeros(16, device=DEV), 8, 8, y)
    torch.cuda.synchronize()


def test_invalid_arguments_rejected_on_host():
    q = torch.zeros(4, 24, dtype=torch.float16, device=DEV)  # K % 16 != 0
    qw = torch.zeros(16, 24, dtype=torch.int8, device=DEV)
    y = torch.empty(4, 16, dtype=torch.float16, device=DEV)
    with pytest.raises(B.OTError) as e:
        B.ot_linear(q, qw, torch.ones(16, device=DEV), torch.zeros(16, device=DEV), 8, 8, y)
    assert e.value.status == B.OT_ERR_INVALID_ARG
    q = torch.zeros(4, 64, dtype=torch.float16, device=DEV)
    qw = torch.zeros(16, 64, dtype=torch.int8, device=DEV)
    with pytest.raises(B.OTError) as e:
        B.ot_linear(q, qw, torch.ones(16, device=DEV), torch.zeros(16, device=DEV), 9, 8, y)
    assert e.value.status == B.OT_ERR_INVALID_ARG
    with pytest.raises(ValueError):
        B.ot_linear(q.cpu(), qw, torch.ones(16, device=DEV), torch.zeros(16, device=DEV), 8, 8, y)


# --------------------------------------------------------------------------
# whole layers of the synthetic OPT workloads
# --------------------------------------------------------------------------
def test_config1_single_linear_full():
    from paper_2406_18832_gb300 import synth
    d = synth.layer_inputs(1, 0, 16)
    g = gpu_layer(d["X_cal"], d["W"], d["b"], d["X"], 8, 8)
    o = oracle_layer(d["X_cal"], d["W"], d["b"], d["X"], 8, 8)
    compare_layer(g, o)


@pytest.mark.parametrize("cfg,li,M,T", [(2, 0, 200, 512), (2, 3, 130, 512), (3, 1, 16, 512), (3, 3, 1, 512),
                                        (3, 2, 128, 512), (4, 1, 64, 256), (5, 2, 96, 256)])
def test_config_layers_reduced_tokens(cfg, li, M, T):
    """Every layer shape family of configs 2-5 at full K and N, fewer tokens."""
    from paper_2406_18832_gb300 import synth
    c = synth.CONFIGS[cfg]
    layer = c.layers[li]
    bits_a, bits_w = c.bits[-1]
    w, b = synth.weights(cfg, li, layer)
    xc = synth.activations(cfg, li, layer, T, 3)
    x = synth.activations(cfg, li, layer, M, 4)
    g = gpu_layer(xc, w, b, x, bits_a, bits_w, relu=layer.relu_out)
    rng = np.random.default_rng(cfg * 10 + li)
    cols = np.sort(rng.choice(layer.N, min(layer.N, 256), replace=False))
    o = oracle_layer(xc, w, b, x, bits_a, bits_w, relu=layer.relu_out, cols=cols)
    compare_layer(g, o, cols=cols)
