"""Asymmetric per-output-channel weights (the paper's "Int8"): the fold, the
code row sums and the corrected linear against the oracle, bit for bit, on
every kernel of the path (decode M <= 16, 16 < M <= 128, prefill M > 128),
with and without the stream-K workspace."""
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


def _gen(seed):
    return torch.Generator().manual_seed(seed)


def _weights(N, K, seed, skew=True):
    g = _gen(seed)
    w = torch.randn(N, K, generator=g) * 0.02
    if skew:
        w[: N // 2] += torch.rand(N // 2, 1, generator=g) * 0.04     # one-sided rows
    return w.half()


def _acts(T, K, seed):
    g = _gen(seed)
    x = torch.randn(T, K, generator=g)
    idx = torch.randperm(K, generator=g)[: max(1, K // 100)]
    x[:, idx] = x[:, idx] * (20 + 60 * torch.rand(idx.numel(), generator=g)) + \
        (-20 + 40 * torch.rand(idx.numel(), generator=g))
    return x.half()


@pytest.mark.parametrize("N,K,bits_w", [(1, 16, 8), (17, 784, 8), (300, 4096, 6), (64, 1040, 4)])
def test_fold_asym_bit_exact(N, K, bits_w):
    from paper_2406_18832_gb300 import binding as B
    x = _acts(256, K, 1 + N)
    w = _weights(N, K, 2 + N)
    b = (torch.randn(N, generator=_gen(3)) * 0.01).half()
    mn, mx = oracle.calibrate(x.numpy())
    z, s, r = oracle.params(mn, mx, 8)
    qw_o, sw_o, zc_o = oracle.fold_codes_asym(w.numpy(), s, bits_w)
    _, _, bf_o = oracle.fold(w.numpy(), b.numpy(), z, s, bits_w)

    d = lambda a, dt=torch.float32: torch.as_tensor(np.asarray(a)).to(dt).to(DEV)
    zg, sg, rg = (torch.empty(K, device=DEV) for _ in range(3))
    qw = torch.empty(N, K, dtype=torch.int8, device=DEV)
    sw = torch.empty(N, device=DEV)
    zc = torch.empty(N, dtype=torch.int32, device=DEV)
    bf = torch.empty(N, device=DEV)
    B.ot_fold_weights_asym(d(mn), d(mx), 8, w.to(DEV), b.to(DEV), bits_w, zg, sg, rg, qw, sw, zc, bf)
    assert np.array_equal(sg.cpu().numpy(), s)
    assert np.array_equal(qw.cpu().numpy(), qw_o)
    assert np.array_equal(sw.cpu().numpy().view(np.uint32), sw_o.view(np.uint32))
    assert np.array_equal(zc.cpu().numpy(), zc_o)
    assert np.array_equal(bf.cpu().numpy().view(np.uint32), bf_o.view(np.uint32))


@pytest.mark.parametrize("M,K", [(1, 8), (3, 768), (65, 4104), (1000, 512), (37, 16392)])
@pytest.mark.parametrize("fmt", ["f16", "i8"])
def test_quantize_rowsum_exact(M, K, fmt):
    from paper_2406_18832_gb300 import binding as B
    x = _acts(M, K, 10 + M)
    cal = _acts(512, K, 11 + K)
    mn, mx = oracle.calibrate(cal.numpy())
    z, s, r = oracle.params(mn, mx, 8)
    q_o = oracle.quantize(x.numpy(), z, r, 8)
    rs_o = oracle.rowsum(q_o)
    f16 = fmt == "f16"
    q = torch.empty(M, K, dtype=torch.float16 if f16 else torch.int8, device=DEV)
    rs = torch.full((M,), 12345, dtype=torch.int32, device=DEV)   # cleared by the call
    B.ot_quantize_act_rowsum(x.to(DEV), torch.as_tensor(z).to(DEV), torch.as_tensor(r).to(DEV), 8, q, rs,
                             B.OT_CODE_F16 if f16 else B.OT_CODE_I8)
    got_q = q.cpu().numpy()
    assert np.array_equal(got_q.astype(np.int64), q_o.astype(np.int64))
    assert np.array_equal(rs.cpu().numpy().astype(np.int64), rs_o)


SHAPES = [(1, 130, 2048), (7, 33, 4112), (16, 777, 2064), (33, 256, 1040), (100, 272, 4096), (128, 128, 1088),
          (200, 500, 640), (300, 1024, 2112)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits", [(8, 8), (6, 6)])
def test_linear_asym_bit_exact(M, N, K, bits):
    from paper_2406_18832_gb300 import binding as B
    ba, bw = bits
    qa = (1 << (ba - 1)) - 1
    q = torch.randint(-qa, qa + 1, (M, K), generator=_gen(M + K), dtype=torch.int32)
    w = _weights(N, K, N + K)
    qw_o, sw_o, zc_o = oracle.fold_codes_asym(w.numpy(), None, bw)
    bf = (torch.randn(N, generator=_gen(N)) * 0.5).float()
    q8 = q.numpy().astype(np.int8)
    acc = oracle.matmul(q8, qw_o)
    rs = oracle.rowsum(q8)
    qd = q.half().to(DEV)
    qwd = torch.as_tensor(qw_o).to(DEV)
    swd = torch.as_tensor(sw_o).to(DEV)
    zcd = torch.as_tensor(zc_o).to(DEV)
    rsd = torch.as_tensor(rs.astype(np.int32)).to(DEV)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    for relu in (False, True):
        ref = oracle.epilogue_asym(acc, rs, zc_o, sw_o, bf.numpy(), relu)
        for workspace in (False, ws, ws):
            y = torch.full((M, N), 7.0, dtype=torch.float16, device=DEV)
            B.ot_linear_asym(qd, qwd, swd, zcd, rsd, bf.to(DEV), ba, bw, y, relu=relu, workspace=workspace)
            torch.cuda.synchronize()
            assert B.ot_get_device_status() == B.OT_OK
            assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))


@pytest.mark.parametrize("M", [4, 100, 300])
def test_linear_asym_extremes(M):
    """Codes at -128 / +127 with zero points at the ends of the range and
    all-+-127 activations: the chunk carries and the int64 correction."""
    from paper_2406_18832_gb300 import binding as B
    N, K = 256, 16384
    q = torch.full((M, K), 127, dtype=torch.int32)
    q[1::3] = -127
    q[2::3, ::2] = -127
    qw = torch.full((N, K), -128, dtype=torch.int32)
    qw[1::2] = 127
    qw[5, K // 2:] = 0
    zc = torch.tensor([(-128 if n % 3 == 0 else (127 if n % 3 == 1 else 3)) for n in range(N)], dtype=torch.int32)
    sw = (torch.rand(N, generator=_gen(5)) * 1e-6).float()
    bf = torch.randn(N, generator=_gen(6)).float()
    q8, qw8 = q.numpy().astype(np.int8), qw.numpy().astype(np.int8)
    acc = oracle.matmul(q8, qw8)
    rs = oracle.rowsum(q8)
    ref = oracle.epilogue_asym(acc, rs, zc.numpy(), sw.numpy(), bf.numpy())
    y = torch.empty(M, N, dtype=torch.float16, device=DEV)
    B.ot_linear_asym(q.half().to(DEV), qw.to(torch.int8).to(DEV), sw.to(DEV), zc.to(DEV),
                     torch.as_tensor(rs.astype(np.int32)).to(DEV), bf.to(DEV), 8, 8, y)
    assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))


def test_asym_layer_end_to_end_and_accuracy():
    """Calibrate, fold with zero points, quantize with row sums, linear: equal
    to the oracle chain, and on one-sided weight rows closer to fp64 XW^T + b
    than the symmetric path (the paper's reason for "Int8")."""
    from paper_2406_18832_gb300 import binding as B
    M, N, K, bits = 64, 256, 1024, 6
    cal, x = _acts(1024, K, 40), _acts(M, K, 41)
    g = _gen(42)
    w = (torch.rand(N, K, generator=g) * 0.03 + 0.005).half()       # one-sided rows
    b = (torch.randn(N, generator=g) * 0.01).half()
    mn, mx = oracle.calibrate(cal.numpy())
    z, s, r = oracle.params(mn, mx, bits)
    qw_o, sw_o, zc_o = oracle.fold_codes_asym(w.numpy(), s, bits)
    qws, sws, bf_o = oracle.fold(w.numpy(), b.numpy(), z, s, bits)
    q_o = oracle.quantize(x.numpy(), z, r, bits)
    ref_asym = oracle.epilogue_asym(oracle.matmul(q_o, qw_o), oracle.rowsum(q_o), zc_o, sw_o, bf_o)
    ref_sym = oracle.epilogue(oracle.matmul(q_o, qws), sws, bf_o)

    d = lambda a: torch.as_tensor(np.asarray(a)).to(DEV)
    zg, sg, rg = (torch.empty(K, device=DEV) for _ in range(3))
    qw = torch.empty(N, K, dtype=torch.int8, device=DEV)
    sw = torch.empty(N, device=DEV)
    zc = torch.empty(N, dtype=torch.int32, device=DEV)
    bf = torch.empty(N, device=DEV)
    B.ot_fold_weights_asym(d(mn), d(mx), bits, w.to(DEV), b.to(DEV), bits, zg, sg, rg, qw, sw, zc, bf)
    q = torch.empty(M, K, dtype=torch.float16, device=DEV)
    rs = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ot_quantize_act_rowsum(x.to(DEV), zg, rg, bits, q, rs)
    y = torch.empty(M, N, dtype=torch.float16, device=DEV)
    B.ot_linear_asym(q, qw, sw, zc, rs, bf, bits, bits, y)
    got = y.cpu().numpy()
    assert np.array_equal(got.view(np.uint16), ref_asym.view(np.uint16))
    exact = x.double().numpy() @ w.double().numpy().T + b.double().numpy()
    err_asym = np.abs(got.astype(np.float64) - exact).mean()
    err_sym = np.abs(ref_sym.astype(np.float64) - exact).mean()
    assert err_asym < err_sym


def test_quantized_linear_asym_layer_matches_oracle():
    """QuantizedLinear(weights="asym"): calibrate, fold, forward == the oracle chain."""
    from paper_2406_18832_gb300 import QuantizedLinear
    M, N, K = 40, 320, 768
    cal, x = _acts(512, K, 60), _acts(M, K, 61)
    w = _weights(N, K, 62)
    b = (torch.randn(N, generator=_gen(63)) * 0.01).half()
    ql = QuantizedLinear(K, N, 8, 8, relu=True, device=DEV, weights="asym")
    ql.calibrate(cal[:256].to(DEV)).calibrate(cal[256:].to(DEV)).fold(w.to(DEV), b.to(DEV))
    y = ql(x.to(DEV)).cpu().numpy()
    mn, mx = oracle.calibrate(cal.numpy())
    z, s, r = oracle.params(mn, mx, 8)
    qw, sw, zc = oracle.fold_codes_asym(w.numpy(), s, 8)
    _, _, bf = oracle.fold(w.numpy(), b.numpy(), z, s, 8)
    q = oracle.quantize(x.numpy(), z, r, 8)
    ref = oracle.epilogue_asym(oracle.matmul(q, qw), oracle.rowsum(q), zc, sw, bf, relu=True)
    assert np.array_equal(y.view(np.uint16), ref.view(np.uint16))
    assert set(ql.state_dict()) >= {"zc", "qw", "sw", "b_fold"}
