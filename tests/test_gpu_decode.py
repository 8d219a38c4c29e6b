"""Decode-sized linears (up to 32 tokens; the weight-streaming kernel takes
M <= 16, the single-CTA tcgen05 kernel 17-32): both against
the oracle, bit for bit, with the workspace (tiles split between CTAs along K,
int32 partials exchanged through it) and without (whole tiles per CTA).

Shapes cover ragged N (not a multiple of the 128-row tile), ragged K (not a
multiple of the 256-wide unit, nor of the 64-wide window), K long enough that
every warp flushes its fp32 chunk sums into int32 several times, tiles split
over up to 128 CTAs, both token-group widths of the weight stream (M <= 8,
M <= 16) and the tcgen05 kernel just above them (17-32 tokens)."""
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


def _codes(shape, qmax, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(-qmax, qmax + 1, shape, generator=g, dtype=torch.int32)


SHAPES = [(1, 16, 16), (1, 33, 4112), (7, 33, 4112), (16, 144, 80), (17, 256, 1040), (32, 96, 5184),
          (1, 64, 32768), (32, 64, 32768), (3, 1000, 16400), (16, 4096, 4096), (31, 300, 131072)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits", [(8, 8), (6, 6)])
def test_decode_s32_bit_exact_split_and_whole(M, N, K, bits):
    from paper_2406_18832_gb300 import binding as B
    ba, bw = bits
    qa, qwm = (1 << (ba - 1)) - 1, (1 << (bw - 1)) - 1
    q = _codes((M, K), qa, 5 * M + K)
    qw = _codes((N, K), qwm, 3 * N + K)
    ref = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    qd, qwd = q.half().to(DEV), qw.to(torch.int8).to(DEV)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    for workspace in (False, ws, ws):  # the second split call reuses the workspace the first left
        acc = torch.full((M, N), -7, dtype=torch.int32, device=DEV)
        B.ot_linear_s32(qd, qwd, ba, bw, acc, workspace=workspace)
        torch.cuda.synchronize()
        assert B.ot_get_device_status() == B.OT_OK
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)


@pytest.mark.parametrize("K", [8192, 16384, 20480])
@pytest.mark.parametrize("workspace", [False, None])
def test_decode_extremes_carry_across_chunks(K, workspace):
    """All-+-127 codes: every warp's fp32 chunk reaches the 2^24 limit and the
    totals need the int32 carry between chunks and between CTAs."""
    from paper_2406_18832_gb300 import binding as B
    M, N = 3, 70
    q = torch.full((M, K), 127, dtype=torch.int32)
    q[1] = -127
    q[2, ::2] = -127
    qw = torch.full((N, K), 127, dtype=torch.int32)
    qw[1::2] = -127
    qw[5, K // 2:] = 1
    acc = torch.empty(M, N, dtype=torch.int32, device=DEV)
    B.ot_linear_s32(q.half().to(DEV), qw.to(torch.int8).to(DEV), 8, 8, acc, workspace=workspace)
    ref = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)


@pytest.mark.parametrize("M,N,K", [(1, 15360, 5120), (16, 5120, 20480), (32, 777, 2064)])
@pytest.mark.parametrize("relu", [False, True])
def test_decode_f16_epilogue_bit_exact(M, N, K, relu):
    """y = fp16(fma(acc, sw, b')) written into a wider row stride, identical
    to the oracle's epilogue; columns past N untouched."""
    from paper_2406_18832_gb300 import binding as B
    q = _codes((M, K), 31, 11 + M)
    qw = _codes((N, K), 31, 13 + N)
    g = torch.Generator().manual_seed(N + K)
    sw = (torch.rand(N, generator=g) * 1e-3).float()
    bf = torch.randn(N, generator=g).float()
    ld = N + 24
    y = torch.full((M, ld), 5.0, dtype=torch.float16, device=DEV)
    B.ot_linear(q.half().to(DEV), qw.to(torch.int8).to(DEV), sw.to(DEV), bf.to(DEV), 6, 6, y[:, :N],
                relu=relu)
    acc = oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))
    ref = oracle.epilogue(acc, sw.numpy(), bf.numpy(), relu)
    got = y.cpu().numpy()
    assert np.array_equal(got[:, :N].view(np.uint16), ref.view(np.uint16))
    assert np.all(got[:, N:] == 5.0)


def test_decode_interleaved_shapes_share_a_workspace():
    """Calls of different shapes in a row on one workspace: each leaves its
    split-tile slots zeroed for the next."""
    from paper_2406_18832_gb300 import binding as B
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    cases = []
    for i, (M, N, K) in enumerate([(4, 64, 32768), (1, 300, 4096), (20, 40, 8704), (4, 64, 32768)]):
        q = _codes((M, K), 127, 100 + i)
        qw = _codes((N, K), 127, 200 + i)
        cases.append((q, qw, oracle.matmul(q.numpy().astype(np.int8), qw.numpy().astype(np.int8))))
    for _ in range(2):
        for q, qw, ref in cases:
            acc = torch.empty(q.shape[0], qw.shape[0], dtype=torch.int32, device=DEV)
            B.ot_linear_s32(q.half().to(DEV), qw.to(torch.int8).to(DEV), 8, 8, acc, workspace=ws)
            assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)
