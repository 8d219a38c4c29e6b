"""ot_linear_fused: the activation quantization (Eq. 6-7) and the linear in one
call, in both forms: the quantize kernel followed by the linear as its
programmatic dependent (OT_FUSE_PDL, the default), and up to 128 tokens the
linear's token producer quantizing X in shared memory (OT_FUSE_PRODUCER:
decode kernel for M <= 16, the single-CTA tcgen05 kernel's token warps for
16 < M <= 128).  Against the oracle
bit for bit on every kernel of the path, with and without the stream-K
workspace, with a strided X, channel counts that end inside a 64-wide
k-block, NaN and infinite inputs, under CUDA-graph capture, and in
back-to-back calls that reuse one code buffer or follow a kernel that
rewrote the weights."""
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


def _acts(T, K, seed):
    g = _gen(seed)
    x = torch.randn(T, K, generator=g)
    idx = torch.randperm(K, generator=g)[: max(1, K // 100)]
    x[:, idx] = x[:, idx] * (20 + 60 * torch.rand(idx.numel(), generator=g)) + \
        (-20 + 40 * torch.rand(idx.numel(), generator=g))
    return x.half()


def _layer(N, K, bits, seed):
    """Calibrated and folded by the oracle: (z, r, qw, sw, b')."""
    cal = _acts(512, K, seed)
    g = _gen(seed + 1)
    w = (torch.randn(N, K, generator=g) * 0.02).half().numpy()
    b = (torch.randn(N, generator=g) * 0.01).half().numpy()
    mn, mx = oracle.calibrate(cal.numpy())
    z, s, r = oracle.params(mn, mx, bits)
    qw, sw, bf = oracle.fold(w, b, z, s, bits)
    return z, r, qw, sw, bf


def _dev(a):
    return torch.as_tensor(np.ascontiguousarray(a)).to(DEV)


SHAPES = [(1, 130, 2048), (7, 33, 4112), (16, 777, 2064), (17, 300, 784), (32, 96, 5184), (33, 256, 1040),
          (64, 4100, 1024), (65, 129, 2000), (100, 272, 4096), (128, 128, 1088), (128, 5120, 20480),
          (200, 500, 640), (300, 1024, 2112)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits", [8, 6])
def test_linear_fused_bit_exact(M, N, K, bits):
    from paper_2406_18832_gb300 import binding as B
    z, r, qw, sw, bf = _layer(N, K, bits, M + N + K)
    x = _acts(M, K + 24, 7 * M + K)                               # strided: ldx = K + 24
    x[0, 3], x[-1, K - 1], x[M // 2, K // 2] = float("nan"), float("inf"), -float("inf")
    xs = x[:, :K]
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    xd = x.to(DEV)[:, :K]
    for relu in (False, True):
        q_o, _, y_o = oracle.linear(np.ascontiguousarray(xs.numpy()), qw, sw, bf, z, r, bits, relu)
        modes = (B.OT_FUSE_AUTO, B.OT_FUSE_PDL) + ((B.OT_FUSE_PRODUCER,) if M <= 128 else ())
        for mode in modes:
            for workspace in (False, ws, ws):
                q = torch.full((M, K), 5.0, dtype=torch.float16, device=DEV)
                y = torch.full((M, N), 7.0, dtype=torch.float16, device=DEV)
                B.ot_linear_fused(xd, _dev(z), _dev(r), bits, _dev(qw), _dev(sw), _dev(bf), bits, q, y, relu=relu,
                                  workspace=workspace, mode=mode)
                torch.cuda.synchronize()
                assert B.ot_get_device_status() == B.OT_OK
                if mode != B.OT_FUSE_PRODUCER:  # the in-producer form writes no codes
                    assert np.array_equal(q.cpu().numpy().astype(np.int64), q_o.astype(np.int64))
                assert np.array_equal(y.cpu().numpy().view(np.uint16), y_o.view(np.uint16)), f"mode {mode}"


@pytest.mark.parametrize("M", [1, 16, 64, 512])
def test_linear_fused_back_to_back_one_code_buffer(M):
    """Five calls in a row on one stream, no synchronization, one code buffer:
    each call's quantization may only start once the previous linear is done
    with the codes, and each linear reads its own call's codes."""
    from paper_2406_18832_gb300 import binding as B
    N, K = 1024, 3072
    z, r, qw, sw, bf = _layer(N, K, 8, 90)
    xs = [_acts(M, K, 100 + i) for i in range(5)]
    q = torch.empty(M, K, dtype=torch.float16, device=DEV)
    ys = [torch.empty(M, N, dtype=torch.float16, device=DEV) for _ in xs]
    args = [_dev(a) for a in (z, r, qw, sw, bf)]
    xd = [x.to(DEV) for x in xs]
    torch.cuda.synchronize()
    for mode in (B.OT_FUSE_PDL,) + ((B.OT_FUSE_PRODUCER,) if M <= 128 else ()):
        for x, y in zip(xd, ys):
            y.fill_(0)
        for x, y in zip(xd, ys):
            B.ot_linear_fused(x, args[0], args[1], 8, args[2], args[3], args[4], 8, q, y, mode=mode)
        torch.cuda.synchronize()
        for x, y in zip(xs, ys):
            _, _, y_o = oracle.linear(x.numpy(), qw, sw, bf, z, r, 8)
            assert np.array_equal(y.cpu().numpy().view(np.uint16), y_o.view(np.uint16))


@pytest.mark.parametrize("M", [4, 96, 400])
def test_linear_fused_after_weight_rewrite(M):
    """The linear reads weights before the quantization ends; weights written
    by kernels earlier on the stream (a copy, the fold) are complete by then."""
    from paper_2406_18832_gb300 import binding as B
    N, K = 640, 2048
    z, r, qw1, sw1, bf = _layer(N, K, 8, 31)
    _, _, qw2, sw2, _ = _layer(N, K, 8, 32)
    x = _acts(M, K, 33)
    qw = _dev(qw1)
    sw = _dev(sw1)
    big = torch.empty(64 << 20, dtype=torch.uint8, device=DEV)
    q = torch.empty(M, K, dtype=torch.float16, device=DEV)
    y = torch.empty(M, N, dtype=torch.float16, device=DEV)
    xd, zd, rd, bfd = x.to(DEV), _dev(z), _dev(r), _dev(bf)
    B.ot_linear_fused(xd, zd, rd, 8, qw, sw, bfd, 8, q, y)
    big.fill_(1)                                                   # a long kernel ahead of the rewrite
    qw.copy_(_dev(qw2))
    sw.copy_(_dev(sw2))
    B.ot_linear_fused(xd, zd, rd, 8, qw, sw, bfd, 8, q, y)
    torch.cuda.synchronize()
    _, _, y_o = oracle.linear(x.numpy(), qw2, sw2, bf, z, r, 8)
    assert np.array_equal(y.cpu().numpy().view(np.uint16), y_o.view(np.uint16))


@pytest.mark.parametrize("M", [1, 16, 256])
def test_linear_fused_in_cuda_graph(M):
    """Captured into a graph (the programmatic dependency becomes a graph
    edge) and replayed on new inputs written into the captured buffers."""
    from paper_2406_18832_gb300 import binding as B
    N, K = 2048, 4096
    z, r, qw, sw, bf = _layer(N, K, 6, 55)
    args = [_dev(a) for a in (z, r, qw, sw, bf)]
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    x = torch.empty(M, K, dtype=torch.float16, device=DEV)
    q = torch.empty(M, K, dtype=torch.float16, device=DEV)
    y = torch.empty(M, N, dtype=torch.float16, device=DEV)
    x.copy_(_acts(M, K, 56).to(DEV))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        B.ot_linear_fused(x, args[0], args[1], 6, args[2], args[3], args[4], 6, q, y, workspace=ws, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        B.ot_linear_fused(x, args[0], args[1], 6, args[2], args[3], args[4], 6, q, y, workspace=ws, stream=s)
    for seed in (57, 58, 59):
        xh = _acts(M, K, seed)
        x.copy_(xh.to(DEV))
        g.replay()
        torch.cuda.synchronize()
        _, _, y_o = oracle.linear(xh.numpy(), qw, sw, bf, z, r, 6)
        assert np.array_equal(y.cpu().numpy().view(np.uint16), y_o.view(np.uint16))
