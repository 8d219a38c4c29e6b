"""LayerNorm fused with the symmetrization and per-channel quantization
(Section 3.2) against the oracle, bit for bit: the folded affine, the codes
(fp16 and int8 formats), the code row sums, and a fused layer end to end."""
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


def _hidden(M, K, seed):
    """Residual-stream-like rows: a per-channel offset, a few large channels,
    rows of very different scale (incl. tiny and near-fp16-max values)."""
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((M, K)) * 2 + rng.standard_normal(K)
    h[:, rng.choice(K, max(1, K // 64), replace=False)] *= 40
    if M >= 4:
        h[1] *= 1e-6                      # subnormal-scale row
        h[2] = np.linspace(-60000, 60000, K)
        h[3] = 0.75                       # constant row: variance 0
    return h.astype(np.float16)


def _affine(K, seed):
    rng = np.random.default_rng(seed)
    gamma = (1 + 0.3 * rng.standard_normal(K)).astype(np.float16)
    beta = (0.2 * rng.standard_normal(K)).astype(np.float16)
    z = (0.5 * rng.standard_normal(K)).astype(np.float32)
    r = (rng.random(K) * 40 + 1).astype(np.float32)
    return gamma, beta, z, r


def test_fold_layernorm_bit_exact():
    from paper_2406_18832_gb300 import binding as B
    K = 1000
    gamma, beta, z, r = _affine(K, 1)
    gr_o, br_o = oracle.fold_layernorm(gamma, beta, z, r)
    t = lambda a: torch.as_tensor(a).to(DEV)
    gr, br = torch.empty(K, device=DEV), torch.empty(K, device=DEV)
    B.ot_fold_layernorm(t(gamma), t(beta), t(z), t(r), gr, br)
    assert np.array_equal(gr.cpu().numpy().view(np.uint32), gr_o.view(np.uint32))
    assert np.array_equal(br.cpu().numpy().view(np.uint32), br_o.view(np.uint32))


@pytest.mark.parametrize("M,K,pad", [(1, 8, 0), (4, 768, 8), (9, 1032, 0), (33, 2048, 8), (65, 4104, 0), (300, 4096, 16),
                                     (7, 9224, 8), (12, 12288, 0), (5, 12296, 0), (6, 36864, 0)])
@pytest.mark.parametrize("fmt", ["f16", "i8"])
@pytest.mark.parametrize("bits", [8, 6])
def test_layernorm_quantize_bit_exact(M, K, pad, fmt, bits):
    from paper_2406_18832_gb300 import binding as B
    h = _hidden(M, K, 10 * M + K)
    gamma, beta, z, r = _affine(K, K)
    gr, br = oracle.fold_layernorm(gamma, beta, z, r)
    eps = 1e-5
    q_o, rs_o, _, _ = oracle.layernorm_quantize(h, gr, br, eps, bits)
    hb = torch.zeros(M, K + pad, dtype=torch.float16)
    hb[:, :K] = torch.as_tensor(h)
    hd = hb.to(DEV)[:, :K]
    f16 = fmt == "f16"
    q = torch.empty(M, K, dtype=torch.float16 if f16 else torch.int8, device=DEV)
    rs = torch.full((M,), -5, dtype=torch.int32, device=DEV)
    B.ot_layernorm_quantize(hd, torch.as_tensor(gr).to(DEV), torch.as_tensor(br).to(DEV), eps, bits, q,
                            B.OT_CODE_F16 if f16 else B.OT_CODE_I8, rowsum=rs)
    assert np.array_equal(q.cpu().numpy().astype(np.int64), q_o.astype(np.int64))
    assert np.array_equal(rs.cpu().numpy().astype(np.int64), rs_o)


def _every_fp16_rows(K, seed):
    """Rows of 2048 values holding every fp16 pattern of one exponent field
    (both signs, all fractions; 31 rows), then every finite fp16 value once
    in a random order over rows of K (zero-padded): each value's split into
    the exact sums, and the sums' range, at least once."""
    rng = np.random.default_rng(seed)
    pats = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    exp = (pats >> 10) & 31
    bands = [rng.permutation(pats[exp == e]) for e in range(31)]
    fin = rng.permutation(pats[exp != 31])
    rows = [np.tile(b, K // 2048) for b in bands]
    allv = np.zeros(-(-fin.size // K) * K, np.uint16)
    allv[: fin.size] = fin
    rows += list(allv.reshape(-1, K))
    return np.stack(rows).view(np.float16)


@pytest.mark.parametrize("K", [2048, 4096, 8192, 12288, 16384, 18432])
@pytest.mark.parametrize("fmt", ["f16", "i8"])
def test_layernorm_quantize_every_fp16_value(K, fmt):
    from paper_2406_18832_gb300 import binding as B
    h = _every_fp16_rows(K, K)
    M = h.shape[0]
    rng = np.random.default_rng(K + 1)
    gr = (30 + rng.standard_normal(K)).astype(np.float32)     # codes mostly inside the 8-bit range
    br = rng.standard_normal(K).astype(np.float32)
    q_o, rs_o, _, _ = oracle.layernorm_quantize(h, gr, br, 0.0, 8)
    f16 = fmt == "f16"
    q = torch.empty(M, K, dtype=torch.float16 if f16 else torch.int8, device=DEV)
    rs = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ot_layernorm_quantize(torch.as_tensor(h).to(DEV), torch.as_tensor(gr).to(DEV), torch.as_tensor(br).to(DEV),
                            0.0, 8, q, B.OT_CODE_F16 if f16 else B.OT_CODE_I8, rowsum=rs)
    got = q.cpu().numpy().astype(np.int64)
    assert np.array_equal(got, q_o.astype(np.int64))
    assert np.array_equal(rs.cpu().numpy().astype(np.int64), rs_o)
    assert np.count_nonzero(np.abs(q_o) == 127) < q_o.size // 4   # the codes are not just saturated


def test_layernorm_quantize_nonfinite_rows_and_no_rowsum():
    from paper_2406_18832_gb300 import binding as B
    M, K = 5, 512
    h = _hidden(M, K, 3)
    h[0, 17] = np.inf
    h[4, 3] = np.nan
    gamma, beta, z, r = _affine(K, 4)
    gr, br = oracle.fold_layernorm(gamma, beta, z, r)
    q_o = oracle.layernorm_quantize(h, gr, br, 0.0, 8)[0]
    q = torch.empty(M, K, dtype=torch.int8, device=DEV)
    B.ot_layernorm_quantize(torch.as_tensor(h).to(DEV), torch.as_tensor(gr).to(DEV), torch.as_tensor(br).to(DEV),
                            0.0, 8, q, B.OT_CODE_I8)
    got = q.cpu().numpy()
    assert np.array_equal(got, q_o)
    assert np.all(got[0] == 0) and np.all(got[4] == 0)


@pytest.mark.parametrize("weights", ["sym", "asym"])
def test_fused_layer_end_to_end(weights):
    """QuantizedLinear: calibrate on LN outputs, fold, fold_layernorm, then
    forward_hidden(h) == the oracle chain (fused codes -> product -> epilogue)."""
    from paper_2406_18832_gb300 import QuantizedLinear
    M, N, K, eps = 64, 384, 1024, 1e-5
    h = _hidden(M, K, 21)
    gamma, beta, _, _ = _affine(K, 22)
    # LN outputs for calibration, in fp64 then fp16 (test data, not the path)
    hc = _hidden(512, K, 23).astype(np.float64)
    ln = (hc - hc.mean(1, keepdims=True)) / np.sqrt(hc.var(1, keepdims=True) + eps) * gamma + beta
    x_cal = ln.astype(np.float16)
    rng = np.random.default_rng(24)
    w = (rng.standard_normal((N, K)) * 0.02 + (0.02 if weights == "asym" else 0)).astype(np.float16)
    b = (rng.standard_normal(N) * 0.01).astype(np.float16)
    ql = QuantizedLinear(K, N, 8, 8, device=DEV, weights=weights)
    ql.calibrate(torch.as_tensor(x_cal).to(DEV)).fold(torch.as_tensor(w).to(DEV), torch.as_tensor(b).to(DEV))
    ql.fold_layernorm(torch.as_tensor(gamma).to(DEV), torch.as_tensor(beta).to(DEV), eps)
    y = ql.forward_hidden(torch.as_tensor(h).to(DEV)).cpu().numpy()

    mn, mx = oracle.calibrate(x_cal)
    z, s, r = oracle.params(mn, mx, 8)
    gr, br = oracle.fold_layernorm(gamma, beta, z, r)
    q, rs, _, _ = oracle.layernorm_quantize(h, gr, br, eps, 8)
    if weights == "asym":
        qw, sw, zc = oracle.fold_codes_asym(w, s, 8)
        _, _, bf = oracle.fold(w, b, z, s, 8)
        ref = oracle.epilogue_asym(oracle.matmul(q, qw), rs, zc, sw, bf)
    else:
        qw, sw, bf = oracle.fold(w, b, z, s, 8)
        ref = oracle.epilogue(oracle.matmul(q, qw), sw, bf)
    assert np.array_equal(y.view(np.uint16), ref.view(np.uint16))
