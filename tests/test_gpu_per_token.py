"""GPU parity of the per-token path (Eq. 3; the paper's out / fc2 linears):
per-token codes and scales, per-output-channel weight codes, int32
accumulators and fp16 outputs, bit for bit against the oracle, through the
decode, small-batch and CTA-pair GEMM kernels."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("M,K,N,bits,relu", [
    (1, 5120, 5120, 6, False), (16, 4096, 4096, 8, False), (33, 768, 768, 8, True), (128, 4096, 4096, 8, False),
    (300, 2112, 1000, 8, False), (2048, 4096, 4096, 8, False), (2048, 16384, 4096, 8, False),
    (1024, 20480, 5120, 6, False)])
def test_per_token_linear_bit_exact(M, K, N, bits, relu):
    from paper_2406_18832_gb300 import binding as B, synth
    dev = "cuda"
    lay = synth.Layer("out", K, N, n_outliers=0)
    x = synth.activations(7, 1, lay, M, 4, device=dev)
    w, b = synth.weights(7, 1, lay, device=dev)
    z_res = torch.randn(N, device=dev) * 0.5          # Eq. 8: residual shift carried in the bias
    bias = b.float() + z_res
    q16 = torch.empty(M, K, dtype=torch.float16, device=dev)
    q8 = torch.empty(M, K, dtype=torch.int8, device=dev)
    s_tok = torch.empty(M, device=dev)
    s_tok8 = torch.empty(M, device=dev)
    B.ot_quantize_tokens(x, bits, q16, s_tok)
    B.ot_quantize_tokens(x, bits, q8, s_tok8, q_format=B.OT_CODE_I8)
    qw = torch.empty(N, K, dtype=torch.int8, device=dev)
    sw = torch.empty(N, device=dev)
    B.ot_quantize_weights(w, bits, qw, sw)
    y = torch.empty(M, N, dtype=torch.float16, device=dev)
    B.ot_linear_per_token(q16, qw, sw, s_tok, bias, bits, bits, y, relu=relu)
    acc = torch.empty(M, N, dtype=torch.int32, device=dev)
    B.ot_linear_s32(q16, qw, bits, bits, acc)
    torch.cuda.synchronize()
    assert B.ot_get_device_status() == B.OT_OK

    rng = np.random.default_rng(M + N)
    rows = np.unique(np.concatenate([[0, M - 1], rng.choice(M, min(M, 24), replace=False)]))
    cols = np.unique(np.concatenate([[0, N - 1], rng.choice(N, min(N, 256), replace=False)]))
    xr = x.cpu().numpy()[rows]
    oq, os_ = oracle.quantize_tokens(xr, bits)
    assert np.array_equal(q8.cpu().numpy()[rows], oq)
    assert np.array_equal(q16.cpu().numpy()[rows].astype(np.int64), oq.astype(np.int64))
    assert np.array_equal(s_tok.cpu().numpy()[rows], os_) and torch.equal(s_tok, s_tok8)
    oqw, osw = oracle.quantize_weights(w.cpu().numpy()[cols], bits)
    assert np.array_equal(qw.cpu().numpy()[cols], oqw) and np.array_equal(sw.cpu().numpy()[cols], osw)
    oacc = oracle.matmul(oq, oqw)
    assert np.array_equal(acc.cpu().numpy()[rows][:, cols].astype(np.int64), oacc)
    oy = oracle.epilogue_tokens(oacc, os_, osw, bias.cpu().numpy()[cols], relu)
    gy = y.cpu().numpy()[rows][:, cols]
    assert np.array_equal(gy.astype(np.float32), oy.astype(np.float32))


def test_per_token_zero_and_nonfinite_rows():
    from paper_2406_18832_gb300 import binding as B
    x = torch.randn(4, 64, dtype=torch.float16)
    x[1] = 0
    x[2, 5] = float("nan")
    x[3, 9] = float("inf")
    q = torch.empty(4, 64, dtype=torch.int8, device="cuda")
    s = torch.empty(4, device="cuda")
    B.ot_quantize_tokens(x.cuda(), 8, q, s, q_format=B.OT_CODE_I8)
    oq, os_ = oracle.quantize_tokens(x.numpy(), 8)
    assert np.array_equal(q.cpu().numpy(), oq) and np.array_equal(s.cpu().numpy(), os_)
    assert os_[1] == 0 and os_[3] == 0
