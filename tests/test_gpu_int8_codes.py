"""int8 activation codes into the product (Eq. 6 with the codes stored as
Int8): ot_quantize_act(OT_CODE_I8) -> ot_linear / ot_linear_s32 with int8
codes, against the oracle bit for bit (int32 accumulators and fp16 outputs)
on every kernel that takes them -- the decode kernel (M <= 16), the
single-CTA tcgen05 kernel's token warps (M > 16, including prefill sizes) --
with and without the stream-K workspace, ragged N, K ending inside a 64-wide
k-block, Int8 and Int6; and the int8 and fp16 code paths give the same bits."""
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


def _case(M, N, K, bits, seed):
    g = torch.Generator().manual_seed(seed)
    cal = torch.randn(256, K, generator=g)
    idx = torch.randperm(K, generator=g)[: max(1, K // 100)]
    cal[:, idx] = cal[:, idx] * 40 + 10
    x = torch.randn(M, K, generator=g)
    x[:, idx] = x[:, idx] * 45 + 10                               # some runtime values saturate
    w = (torch.randn(N, K, generator=g) * 0.02).half().numpy()
    b = (torch.randn(N, generator=g) * 0.01).half().numpy()
    mn, mx = oracle.calibrate(cal.half().numpy())
    z, s, r = oracle.params(mn, mx, bits)
    qw, sw, bf = oracle.fold(w, b, z, s, bits)
    return x.half(), z, r, qw, sw, bf


def _d(a):
    return torch.as_tensor(np.ascontiguousarray(a)).to(DEV)


SHAPES = [(1, 777, 2064), (9, 5120, 20480), (16, 130, 4112), (17, 96, 5184), (64, 1000, 1040),
          (100, 384, 4096), (128, 5120, 20480), (129, 272, 2112), (300, 1024, 4096), (2048, 4096, 4096)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits", [8, 6])
def test_int8_codes_bit_exact(M, N, K, bits):
    from paper_2406_18832_gb300 import binding as B
    x, z, r, qw, sw, bf = _case(M, N, K, bits, M * 7 + N + K + bits)
    oq = oracle.quantize(x.numpy(), z, r, bits)
    oacc = oracle.matmul_mt(oq, qw)
    oy = oracle.epilogue_mt(oacc, sw, bf, False)
    xd, zd, rd, qwd, swd, bfd = _d(x), _d(z), _d(r), _d(qw), _d(sw), _d(bf)
    q8 = torch.empty(M, K, dtype=torch.int8, device=DEV)
    q16 = torch.empty(M, K, dtype=torch.float16, device=DEV)
    B.ot_quantize_act(xd, zd, rd, bits, q8, B.OT_CODE_I8)
    B.ot_quantize_act(xd, zd, rd, bits, q16, B.OT_CODE_F16)
    torch.cuda.synchronize()
    assert np.array_equal(q8.cpu().numpy(), oq)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    for workspace in (False, ws, ws):
        y = torch.full((M, N), 3.0, dtype=torch.float16, device=DEV)
        acc = torch.full((M, N), 7, dtype=torch.int32, device=DEV)
        B.ot_linear(q8, qwd, swd, bfd, bits, bits, y, workspace=workspace)
        B.ot_linear_s32(q8, qwd, bits, bits, acc, workspace=workspace)
        torch.cuda.synchronize()
        assert B.ot_get_device_status() == B.OT_OK
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), oacc), "int32 accumulators"
        assert np.array_equal(y.cpu().numpy().view(np.uint16), oy.view(np.uint16)), "fp16 outputs"
    y16 = torch.empty(M, N, dtype=torch.float16, device=DEV)
    B.ot_linear(q16, qwd, swd, bfd, bits, bits, y16, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(y16, y)


def test_int8_codes_extremes():
    """All codes and weights at +-qmax: the largest exact partial sums."""
    from paper_2406_18832_gb300 import binding as B
    for M, N, K in [(1, 256, 20480), (40, 512, 20480), (200, 256, 8192)]:
        g = torch.Generator().manual_seed(M)
        q = (torch.randint(0, 2, (M, K), generator=g) * 254 - 127).to(torch.int8)
        qw = (torch.randint(0, 2, (N, K), generator=g) * 254 - 127).to(torch.int8)
        acc = torch.empty(M, N, dtype=torch.int32, device=DEV)
        B.ot_linear_s32(q.to(DEV), qw.to(DEV), 8, 8, acc)
        torch.cuda.synchronize()
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), oracle.matmul_mt(q.numpy(), qw.numpy()))
