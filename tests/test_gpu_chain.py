"""The chained epilogue (Section 3.2 fuses each activation quantization into
the kernel that produces the activation): fc1's epilogue, ReLU included,
writes fc2's activation codes round((v - z') * r') instead of its fp16
output.  Against the oracle bit for bit on every kernel of the path (decode
M <= 16, 16 < M <= 128, prefill M > 128), with and without the stream-K
workspace, on cases built to land on exact rounding ties, and at the full
size of an OPT-30B block's fc1 on sampled rows."""
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


def _codes(shape, qmax, seed):
    return torch.randint(-qmax, qmax + 1, shape, generator=_gen(seed), dtype=torch.int32)


def _next_params(v, bits_next, seed):
    """z', r' of a next layer calibrated on v (per column), as Eq. 3 and 4 give
    them, with a random shrink so that some codes clip."""
    mn, mx = v.min(axis=0), v.max(axis=0)
    z = ((mx + mn) / 2).astype(np.float32)
    qm = (1 << (bits_next - 1)) - 1
    span = np.maximum((mx - mn) / 2, 1e-3)
    shrink = 0.8 + 0.4 * np.random.default_rng(seed).random(v.shape[1])
    r = (qm / (span * shrink)).astype(np.float32)
    return z, r


SHAPES = [(1, 130, 2048), (7, 33, 4112), (16, 777, 2064), (32, 96, 5184), (33, 256, 1040), (100, 272, 4096),
          (128, 128, 1088), (200, 500, 640), (300, 1024, 2112), (1000, 384, 1024)]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("bits,bits_next", [((8, 8), 8), ((6, 6), 6), ((8, 8), 4)])
def test_linear_quantize_next_bit_exact(M, N, K, bits, bits_next):
    from paper_2406_18832_gb300 import binding as B
    ba, bw = bits
    qa, qwm = (1 << (ba - 1)) - 1, (1 << (bw - 1)) - 1
    q = _codes((M, K), qa, M + K)
    qw = _codes((N, K), qwm, 3 * N + K + 1).numpy().astype(np.int8)   # not q's seed when M == N
    sw = (torch.rand(N, generator=_gen(N)) * 1e-4 + 1e-6).float().numpy()
    bf = (torch.randn(N, generator=_gen(N + 1)) * 0.5).float().numpy()
    acc = oracle.matmul(q.numpy().astype(np.int8), qw)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    d = lambda a: torch.as_tensor(np.ascontiguousarray(a)).to(DEV)
    qd, qwd, swd, bfd = q.half().to(DEV), d(qw), d(sw), d(bf)
    for relu in (False, True):
        v = oracle.epilogue(acc, sw, bf, relu).astype(np.float32)
        zn, rn = _next_params(v, bits_next, M + N + K)
        ref = oracle.epilogue_quantize(acc, sw, bf, zn, rn, bits_next, relu)
        assert np.unique(ref).size > 8
        for workspace in (False, ws, ws):
            out = torch.full((M, N), 99.0, dtype=torch.float16, device=DEV)
            B.ot_linear_quantize_next(qd, qwd, swd, bfd, ba, bw, d(zn), d(rn), bits_next, out, relu=relu,
                                      workspace=workspace)
            torch.cuda.synchronize()
            assert B.ot_get_device_status() == B.OT_OK
            got = out.cpu().numpy()
            assert np.array_equal(got, np.round(got))           # fp16 integers
            assert np.array_equal(got.astype(np.int64), ref.astype(np.int64))


@pytest.mark.parametrize("M", [5, 64, 256])
def test_linear_quantize_next_ties_round_half_even(M):
    """sw = 2^-7, b' = j / 128, z' = 0, r' = 64: (v - z') r' = (acc + j) / 2 is
    exact and a tie whenever acc + j is odd -- half the outputs.  Round half
    away from zero, or rounding the fp16 v first, fails here."""
    from paper_2406_18832_gb300 import binding as B
    N, K = 384, 1024
    q = _codes((M, K), 1, 70 + M)                                  # small codes: u stays in range
    qw = _codes((N, K), 1, 71).numpy().astype(np.int8)
    acc = oracle.matmul(q.numpy().astype(np.int8), qw)
    assert np.abs(acc).max() < 2 ** 16
    sw = np.full(N, 2.0 ** -7, np.float32)
    bf = (np.arange(N) % 9 - 4).astype(np.float32) / 128
    zn = np.zeros(N, np.float32)
    rn = np.full(N, 64.0, np.float32)
    ref = oracle.epilogue_quantize(acc, sw, bf, zn, rn, 8, relu=True)
    u = (acc + np.arange(N) % 9 - 4) / 2
    assert np.mean((u != np.floor(u)) & (u > 0) & (u < 127)) > 0.15   # many positive ties in range
    out = torch.empty(M, N, dtype=torch.float16, device=DEV)
    d = lambda a: torch.as_tensor(np.ascontiguousarray(a)).to(DEV)
    B.ot_linear_quantize_next(q.half().to(DEV), d(qw), d(sw), d(bf), 4, 4, d(zn), d(rn), 8, out, relu=True)
    assert np.array_equal(out.cpu().numpy().astype(np.int64), ref.astype(np.int64))


def test_block_fused_chain_matches_oracle_and_unfused():
    """QuantizedBlockLinears.forward(fused=True): fc2's codes come out of fc1's
    epilogue.  They equal the oracle's chained epilogue on fc1's accumulators,
    and differ from quantizing the fp16 f of the unfused path by at most one
    and only where the fp16 rounding of f moved a value across a tie."""
    from paper_2406_18832_gb300 import QuantizedBlockLinears, binding
    h, ffn, T, M = 256, 1024, 2048, 300
    g = _gen(5)
    weights = []
    for K, N in ((h, 3 * h), (h, h), (h, ffn), (ffn, h)):
        weights.append(((torch.randn(N, K, generator=g) / K ** 0.5).half().to(DEV),
                        (torch.randn(N, generator=g) * 0.05).half().to(DEV)))
    x_cal = (torch.randn(T, h, generator=g) * (1 + 8 * torch.rand(h, generator=g))).half().to(DEV)
    x = (torch.randn(M, h, generator=g) * (1 + 8 * torch.rand(h, generator=g))).half().to(DEV)
    blk = QuantizedBlockLinears(h, ffn, 8, 8, device=DEV).calibrate(x_cal, weights)
    plain = blk.forward(x)
    fused = blk.forward(x, fused=True)
    torch.cuda.synchronize()
    assert binding.ot_get_device_status() == binding.OT_OK
    assert torch.equal(plain["o"], fused["o"])
    q1 = blk.fc1.quantize(fused["o"]).cpu().numpy().astype(np.int8)
    acc = oracle.matmul(q1, blk.fc1.qw.cpu().numpy())
    ref = oracle.epilogue_quantize(acc, blk.fc1.sw.cpu().numpy(), blk.fc1.b_fold.cpu().numpy(),
                                   blk.fc2.z.cpu().numpy(), blk.fc2.r.cpu().numpy(), 8, relu=True)
    qf = fused["qf"].cpu().numpy().astype(np.int64)
    assert np.array_equal(qf, ref.astype(np.int64))
    q2 = blk.fc2.quantize(plain["f"]).cpu().numpy().astype(np.int64)
    diff = qf != q2
    assert np.abs(qf - q2).max() <= 1 and diff.mean() < 0.05
    # the fused y is fc2 on those codes: bit-exact against the oracle epilogue
    y_ref = oracle.epilogue(oracle.matmul(qf.astype(np.int8), blk.fc2.qw.cpu().numpy()),
                            blk.fc2.sw.cpu().numpy(), blk.fc2.b_fold.cpu().numpy())
    assert np.array_equal(fused["y"].cpu().numpy().view(np.uint16), y_ref.view(np.uint16))


@pytest.mark.parametrize("M", [16, 4096])
def test_full_size_opt30b_fc1_chained_sampled(M):
    """OPT-30B's fc1 (7168 -> 28672, ReLU) writing fc2's codes at the block
    benchmark's token count: sampled rows and columns against the oracle."""
    from paper_2406_18832_gb300 import QuantizedLinear, synth
    c = synth.CONFIGS[5]
    l1, l2 = c.layers[2], c.layers[3]
    w1, b1 = synth.weights(5, 2, l1, device=DEV)
    w2, b2 = synth.weights(5, 3, l2, device=DEV)
    xc = synth.activations(5, 2, l1, 4096, 3, device=DEV)
    x = synth.activations(5, 2, l1, M, 4, device=DEV)
    fc1 = QuantizedLinear(l1.K, l1.N, 8, 8, relu=True, device=DEV)
    fc2 = QuantizedLinear(l2.K, l2.N, 8, 8, device=DEV)
    fc1.calibrate(xc).fold(w1, b1)
    fc2.calibrate(fc1(xc)).fold(w2, b2)
    q = fc1.quantize(x)
    qf = fc1.linear_quantize_next(q, fc2)
    torch.cuda.synchronize()
    rng = np.random.default_rng(M)
    rows = np.unique(np.concatenate([[0, M - 1], rng.choice(M, min(M, 12), replace=False)]))
    rows_t = torch.from_numpy(rows).to(DEV)
    qr = q.index_select(0, rows_t).cpu().numpy().astype(np.int8)
    acc = oracle.matmul(qr, fc1.qw.cpu().numpy())
    ref = oracle.epilogue_quantize(acc, fc1.sw.cpu().numpy(), fc1.b_fold.cpu().numpy(), fc2.z.cpu().numpy(),
                                   fc2.r.cpu().numpy(), 8, relu=True)
    assert np.array_equal(qf.index_select(0, rows_t).cpu().numpy().astype(np.int64), ref.astype(np.int64))
    assert bool((qf.abs() <= 127).all()) and bool(torch.equal(qf, qf.round()))
