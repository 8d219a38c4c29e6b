"""Stream-K scheduling of the prefill GEMM (a zero-filled workspace lets the
CTA pairs split tiles along K and exchange exact int32 partial sums) gives
results bit-identical to whole-tile scheduling and to the oracle, over
repeated calls that reuse the workspace."""
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


def _codes(shape, qmax, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(-qmax, qmax + 1, shape, generator=g, dtype=torch.int32)


@pytest.mark.parametrize("M,N,K", [(2048, 12288, 4096), (2048, 4096, 4096), (2048, 4096, 16384),
                                   (256, 512, 4096), (300, 1000, 2112), (4096, 256, 1024), (129, 256, 64),
                                   # fewer tiles than CTAs or pairs, split when a fifth / a third shorter
                                   (32, 12288, 4096), (64, 15360, 5120), (100, 12288, 4096)])
def test_streamk_equals_whole_tiles(M, N, K):
    from paper_2406_18832_gb300 import binding as B
    dev = "cuda"
    q = _codes((M, K), 127, M + N).half().to(dev)
    qw = _codes((N, K), 127, K).to(torch.int8).to(dev)
    a_plain = torch.empty(M, N, dtype=torch.int32, device=dev)
    a_sk = torch.empty(M, N, dtype=torch.int32, device=dev)
    B.ot_linear_s32(q, qw, 8, 8, a_plain, workspace=False)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    for _ in range(3):  # the workspace is reused across calls
        a_sk.fill_(-1)
        B.ot_linear_s32(q, qw, 8, 8, a_sk, workspace=ws)
        torch.cuda.synchronize()
        assert B.ot_get_device_status() == B.OT_OK
        assert torch.equal(a_sk, a_plain)
    sw = torch.rand(N, device=dev) * 1e-4
    bf = torch.randn(N, device=dev)
    y1 = torch.empty(M, N, dtype=torch.float16, device=dev)
    y2 = torch.empty(M, N, dtype=torch.float16, device=dev)
    B.ot_linear(q, qw, sw, bf, 8, 8, y1, workspace=False)
    B.ot_linear(q, qw, sw, bf, 8, 8, y2, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
    rng = np.random.default_rng(M * 7 + N)
    rows = rng.choice(M, min(M, 16), replace=False)
    cols = rng.choice(N, min(N, 64), replace=False)
    ref = oracle.matmul(q.cpu().numpy()[rows].astype(np.int8), qw.cpu().numpy()[cols])
    got = a_sk.cpu().numpy()[rows][:, cols].astype(np.int64)
    assert np.array_equal(got, ref)


def test_workspace_size_is_stable():
    from paper_2406_18832_gb300 import binding as B
    n = B.ot_linear_workspace_size()
    assert n > 0 and n == B.ot_linear_workspace_size()


@pytest.mark.parametrize("M,N,K", [(1, 5120, 20480), (16, 2048, 4096), (2048, 4096, 16384), (256, 512, 4096)])
def test_streamk_under_cuda_graph_replay(M, N, K):
    """A captured call replayed many times: each replay must take a new launch
    epoch on the device (one fixed at capture would let a finisher read the
    previous replay's partial sums).  Inputs change between replays; every
    replay is checked against whole-tile scheduling of the same inputs."""
    from paper_2406_18832_gb300 import binding as B
    dev = "cuda"
    qw = _codes((N, K), 127, K + 1).to(torch.int8).to(dev)
    q = torch.empty(M, K, dtype=torch.float16, device=dev)
    acc = torch.empty(M, N, dtype=torch.int32, device=dev)
    want = torch.empty(M, N, dtype=torch.int32, device=dev)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    s = torch.cuda.Stream()
    q.copy_(_codes((M, K), 127, 1).half().to(dev))
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        B.ot_linear_s32(q, qw, 8, 8, acc, workspace=ws, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        B.ot_linear_s32(q, qw, 8, 8, acc, workspace=ws, stream=s)
    for seed in range(2, 8):
        q.copy_(_codes((M, K), 127, seed).half().to(dev))
        acc.fill_(-7)
        g.replay()
        B.ot_linear_s32(q, qw, 8, 8, want, workspace=False)
        torch.cuda.synchronize()
        assert B.ot_get_device_status() == B.OT_OK
        assert torch.equal(acc, want), seed


@pytest.mark.parametrize("M,N,K", [(129, 1, 128), (193, 257, 384), (256, 512, 640), (385, 1024, 4224),
                                   (512, 1024, 2176), (700, 2048, 896)])
def test_pair_kernel_groups_and_ragged_edges(M, N, K):
    """The prefill kernel (M > 128, K % 128 == 0) loads four k-blocks per copy:
    K of 2, 6, 10, 66, 34 and 14 k-blocks (last group short), stream-K pieces
    that start at odd k-blocks, one-row and one-column tails, N = 1.  Against
    the oracle's int64 product, with and without the workspace."""
    from paper_2406_18832_gb300 import binding as B
    dev = "cuda"
    q = _codes((M, K), 127, 3 * M + K)
    qw = _codes((N, K), 127, 5 * N + K).to(torch.int8)
    want = oracle.matmul(q.numpy().astype(np.int8), qw.numpy())
    qd, qwd = q.half().to(dev), qw.to(dev)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
    for workspace in (False, ws, ws):
        acc = torch.full((M, N), -3, dtype=torch.int32, device=dev)
        B.ot_linear_s32(qd, qwd, 8, 8, acc, workspace=workspace)
        torch.cuda.synchronize()
        assert B.ot_get_device_status() == B.OT_OK
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
