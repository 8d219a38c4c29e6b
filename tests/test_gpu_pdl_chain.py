"""Consecutive linears on one stream launch as programmatic dependents of one
another: each may start while the one before it finishes, and must read the
codes that one writes only after it has ended.  A chain of three linears in
which the first two write the next one's codes in their epilogue
(fc1 -> ReLU -> codes -> fc2 -> codes -> fc3), issued back to back for several
inputs without synchronizing, and replayed from a CUDA graph, against the
oracle bit for bit, at decode, mid and prefill token counts, with the
stream-K workspace shared by every call."""
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


def _layer(K, N, bits, g):
    w = (torch.randn(N, K, generator=g) * 0.03).half().numpy()
    b = (torch.randn(N, generator=g) * 0.1).half().numpy()
    cal = (torch.randn(128, K, generator=g) * 2).half().numpy()
    z, s, r = oracle.params(*oracle.calibrate(cal), bits)
    qw, sw, bf = oracle.fold(w, b, z, s, bits)
    return dict(z=z, r=r, qw=qw, sw=sw, bf=bf)


def _d(a):
    return torch.as_tensor(np.ascontiguousarray(a)).to(DEV)


@pytest.mark.parametrize("M", [1, 16, 100, 300])
def test_chained_linears_back_to_back_and_in_a_graph(M):
    from paper_2406_18832_gb300 import binding as B
    g = torch.Generator().manual_seed(M)
    K0, N1, N2, N3, bits = 1024, 2048, 1536, 768, 8
    L1, L2, L3 = _layer(K0, N1, bits, g), _layer(N1, N2, bits, g), _layer(N2, N3, bits, g)
    D = [{k: _d(v) for k, v in L.items()} for L in (L1, L2, L3)]
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    xs = [(torch.randn(M, K0, generator=g) * 2).half() for _ in range(4)]

    def oracle_chain(x):
        q1 = oracle.quantize(x.numpy(), L1["z"], L1["r"], bits)
        q2 = oracle.epilogue_quantize(oracle.matmul(q1, L1["qw"]), L1["sw"], L1["bf"], L2["z"], L2["r"], bits, True)
        q3 = oracle.epilogue_quantize(oracle.matmul(q2, L2["qw"]), L2["sw"], L2["bf"], L3["z"], L3["r"], bits, True)
        return oracle.epilogue(oracle.matmul(q3, L3["qw"]), L3["sw"], L3["bf"])

    xd = torch.empty(M, K0, dtype=torch.float16, device=DEV)
    q1 = torch.empty(M, K0, dtype=torch.float16, device=DEV)
    q2 = torch.empty(M, N1, dtype=torch.float16, device=DEV)
    q3 = torch.empty(M, N2, dtype=torch.float16, device=DEV)

    def chain(y, stream=None):
        B.ot_quantize_act(xd, D[0]["z"], D[0]["r"], bits, q1, B.OT_CODE_F16, stream=stream)
        B.ot_linear_quantize_next(q1, D[0]["qw"], D[0]["sw"], D[0]["bf"], bits, bits, D[1]["z"], D[1]["r"], bits, q2,
                                  relu=True, workspace=ws, stream=stream)
        B.ot_linear_quantize_next(q2, D[1]["qw"], D[1]["sw"], D[1]["bf"], bits, bits, D[2]["z"], D[2]["r"], bits, q3,
                                  relu=True, workspace=ws, stream=stream)
        B.ot_linear(q3, D[2]["qw"], D[2]["sw"], D[2]["bf"], bits, bits, y, workspace=ws, stream=stream)

    # back to back: each input copied in, chained, nothing synchronized until the end
    ys = [torch.empty(M, N3, dtype=torch.float16, device=DEV) for _ in xs]
    for x, y in zip(xs, ys):
        xd.copy_(x.to(DEV), non_blocking=True)
        chain(y)
    torch.cuda.synchronize()
    assert B.ot_get_device_status() == B.OT_OK
    refs = [oracle_chain(x) for x in xs]
    for y, ref in zip(ys, refs):
        assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))

    # captured once, replayed on new inputs
    s = torch.cuda.Stream()
    y = torch.empty(M, N3, dtype=torch.float16, device=DEV)
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        chain(y, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        chain(y, stream=s)
    for x, ref in zip(xs[::-1], refs[::-1]):
        xd.copy_(x.to(DEV))
        graph.replay()
        torch.cuda.synchronize()
        assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16))


@pytest.mark.parametrize("M", [1, 16, 100, 300])
def test_fused_call_reads_weights_folded_just_before(M):
    """ot_linear_fused loads its first weights before the codes are ready
    (decode: into its ring): the quantize kernel in front of it waits for the
    kernel before it and only then releases the linear.  Two weight sets are
    folded alternately into the same buffers, each fold followed at once by a
    fused call on the same stream, nothing synchronized in between: every
    output must be the oracle's for the weights folded just before it."""
    from paper_2406_18832_gb300 import binding as B
    g = torch.Generator().manual_seed(500 + M)
    K, N, bits = 2048, 3072, 8
    cal = (torch.randn(256, K, generator=g) * 2).half().numpy()
    mn, mx = oracle.calibrate(cal)
    z, s, r = oracle.params(mn, mx, bits)
    ws_h = [(torch.randn(N, K, generator=g) * 0.03).half().numpy() for _ in range(2)]
    bs_h = [(torch.randn(N, generator=g) * 0.1).half().numpy() for _ in range(2)]
    folds = [oracle.fold(w, b, z, s, bits) for w, b in zip(ws_h, bs_h)]
    xs = [(torch.randn(M, K, generator=g) * 2).half() for _ in range(6)]
    refs = [oracle.linear(x.numpy(), *folds[i % 2], z, r, bits)[2] for i, x in enumerate(xs)]

    dmn, dmx = _d(mn), _d(mx)
    dz, ds, dr = (torch.empty(K, device=DEV) for _ in range(3))
    qw = torch.empty(N, K, dtype=torch.int8, device=DEV)
    sw, bf = torch.empty(N, device=DEV), torch.empty(N, device=DEV)
    dw = [_d(w) for w in ws_h]
    db = [_d(b) for b in bs_h]
    dx = [x.to(DEV) for x in xs]
    q = torch.empty(M, K, dtype=torch.float16, device=DEV)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    ys = [torch.empty(M, N, dtype=torch.float16, device=DEV) for _ in xs]
    torch.cuda.synchronize()
    for i, (x, y) in enumerate(zip(dx, ys)):
        B.ot_fold_weights(dmn, dmx, bits, dw[i % 2], db[i % 2], bits, dz, ds, dr, qw, sw, bf)
        B.ot_linear_fused(x, dz, dr, bits, qw, sw, bf, bits, q, y, workspace=ws)
    torch.cuda.synchronize()
    assert B.ot_get_device_status() == B.OT_OK
    for i, (y, ref) in enumerate(zip(ys, refs)):
        assert np.array_equal(y.cpu().numpy().view(np.uint16), ref.view(np.uint16)), f"call {i}"
