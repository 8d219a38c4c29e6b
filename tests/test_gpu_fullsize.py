"""GPU parity at the workloads' full sizes (the launch configurations the
benchmark times), against the oracle on the same seeded inputs.

Per layer, on the GPU and in the oracle:
  - calibration over the configuration's 65,536 calibration tokens, streamed in
    blocks of 8192 through both sides: every channel's min / max;
  - every z, s, r;
  - the whole fold: every weight code, every sw and every b';
  - for each token count: every activation code, and the int32 accumulators
    and fp16 outputs -- all of them where the oracle's product finishes in
    seconds (configs 1 and 2, config 3 up to 128 tokens), else on a sample of
    rows and columns that meets every token tile of the tcgen05 kernels (64-,
    96-, 128- and 192-row tiles, first and last row of each) and every 128-row
    weight tile (first and last channel of each, and of each 32-lane quarter),
    so every (token tile, weight tile) pair -- stream-K split tiles included,
    whose accumulators hold every k-range -- contributes outputs.
The int8-code input and the fused call (quantization inside the linear up to
128 tokens) must give the same bits as the checked output.  The oracle runs
its C functions over row ranges in host threads (identical arithmetic,
bit-identical results)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_f16_close

pytestmark = pytest.mark.gpu

CAL_TOKENS = 65536
CHUNK = 8192


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _tile_rows(M: int, rng) -> np.ndarray:
    """Rows meeting every 64/96/128/192-row token tile at both ends, plus random rows."""
    r = [0, M - 1]
    for t in (64, 96, 128, 192):
        for t0 in range(0, M, t):
            r += [t0, min(M, t0 + t) - 1]
    r += list(rng.choice(M, min(M, 64), replace=False))
    return np.unique(np.asarray(r, dtype=np.int64))


def _tile_cols(N: int, rng, per_tile: int = 12) -> np.ndarray:
    """Channels meeting every 128-row weight tile (ends of the tile and of each
    32-lane quarter) plus random channels of every tile."""
    c = []
    for n0 in range(0, N, 128):
        n1 = min(N, n0 + 128)
        c += [n for n in (n0, n0 + 31, n0 + 32, n0 + 63, n0 + 64, n0 + 95, n0 + 96, n1 - 1) if n < n1]
        c += list(n0 + rng.choice(n1 - n0, min(n1 - n0, per_tile), replace=False))
    return np.unique(np.asarray(c, dtype=np.int64))


def _build_layer(cfg, li, bits):
    """GPU layer (calibrated on 65,536 tokens, folded) and the oracle's artefact, compared in full."""
    from paper_2406_18832_gb300 import QuantizedLinear, synth
    dev = torch.device("cuda")
    layer = synth.CONFIGS[cfg].layers[li]
    bits_a, bits_w = bits
    T = min(CAL_TOKENS, synth.CONFIGS[cfg].T_cal)
    w, b = synth.weights(cfg, li, layer, device=dev)
    ql = QuantizedLinear(layer.K, layer.N, bits_a, bits_w, relu=layer.relu_out, device=dev)
    mn = mx = None
    for blk in synth.activation_chunks(cfg, li, layer, T, 3, device=dev, chunk=CHUNK):
        ql.calibrate(blk)
        mn, mx = oracle.calibrate_mt(blk.cpu().numpy(), mn, mx)
    ql.fold(w, b)
    torch.cuda.synchronize()
    z, s, r = oracle.params(mn, mx, bits_a)
    assert np.array_equal(ql.ch_min.cpu().numpy(), mn) and np.array_equal(ql.ch_max.cpu().numpy(), mx)
    assert np.array_equal(ql.z.cpu().numpy(), z) and np.array_equal(ql.s.cpu().numpy(), s)
    assert np.array_equal(ql.r.cpu().numpy(), r)
    qw, sw, bf = oracle.fold_mt(w.cpu().numpy(), b.cpu().numpy(), z, s, bits_w)
    assert np.array_equal(ql.qw.cpu().numpy(), qw), "weight codes"
    assert np.array_equal(ql.sw.cpu().numpy(), sw), "sw"
    assert np.array_equal(ql.b_fold.cpu().numpy(), bf), "b'"
    return layer, ql, dict(z=z, r=r, qw=qw, sw=sw, bf=bf)


def _check_tokens(cfg, li, layer, ql, o, M, bits, full: bool):
    from paper_2406_18832_gb300 import binding, synth
    dev = torch.device("cuda")
    bits_a, bits_w = bits
    x = synth.activations(cfg, li, layer, M, 4, device=dev)
    q = ql.quantize(x)
    y = ql.linear(q)
    acc = torch.empty(M, layer.N, dtype=torch.int32, device=dev)
    binding.ot_linear_s32(q, ql.qw, bits_a, bits_w, acc)
    torch.cuda.synchronize()
    assert binding.ot_get_device_status() == binding.OT_OK

    oq = oracle.quantize_mt(x.cpu().numpy(), o["z"], o["r"], bits_a)
    assert np.array_equal(q.cpu().numpy().astype(np.int64), oq.astype(np.int64)), f"codes M={M}"
    if full:
        oacc = oracle.matmul_mt(oq, o["qw"])
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), oacc), f"int32 accumulators M={M}"
        oy = oracle.epilogue_mt(oacc, o["sw"], o["bf"], layer.relu_out)
        gy = y.cpu().numpy()
    else:
        rng = np.random.default_rng(cfg * 1000 + li * 10 + M)
        rows, cols = _tile_rows(M, rng), _tile_cols(layer.N, rng)
        oacc = oracle.matmul_mt(oq[rows], o["qw"][cols])
        gacc = acc.cpu().numpy()[np.ix_(rows, cols)].astype(np.int64)
        assert np.array_equal(gacc, oacc), f"int32 accumulators M={M} ({len(rows)} x {len(cols)} sample)"
        oy = oracle.epilogue_mt(oacc, o["sw"][cols], o["bf"][cols], layer.relu_out)
        gy = y.cpu().numpy()[np.ix_(rows, cols)]
        assert torch.isfinite(y).all()
        if layer.relu_out:
            assert (y >= 0).all()
    assert_f16_close(gy, oy, what=f"y M={M}")
    # one fp32 fma rounded once to fp16 on both sides: bit-identical
    assert np.array_equal(gy.view(np.uint16), oy.view(np.uint16)), f"fp16 outputs M={M}"

    # the same layer from int8 codes, and with the quantization inside the
    # linear (ot_linear_fused): the same bits as the checked output
    q8 = torch.empty(M, layer.K, dtype=torch.int8, device=dev)
    binding.ot_quantize_act(x, ql.z, ql.r, bits_a, q8, binding.OT_CODE_I8)
    y8 = torch.empty_like(y)
    binding.ot_linear(q8, ql.qw, ql.sw, ql.b_fold, bits_a, bits_w, y8, relu=layer.relu_out)
    yf = torch.empty_like(y)
    binding.ot_linear_fused(x, ql.z, ql.r, bits_a, ql.qw, ql.sw, ql.b_fold, bits_w, torch.empty_like(q), yf,
                            relu=layer.relu_out)
    yp = None
    if M <= 128:
        yp = torch.empty_like(y)
        binding.ot_linear_fused(x, ql.z, ql.r, bits_a, ql.qw, ql.sw, ql.b_fold, bits_w, torch.empty_like(q), yp,
                                relu=layer.relu_out, mode=binding.OT_FUSE_PRODUCER)
    torch.cuda.synchronize()
    assert binding.ot_get_device_status() == binding.OT_OK
    assert np.array_equal(q8.cpu().numpy(), oq), f"int8 codes M={M}"
    assert torch.equal(y8, y), f"int8-code linear M={M}"
    assert torch.equal(yf, y), f"fused linear M={M}"
    assert yp is None or torch.equal(yp, y), f"linear quantizing in its producer M={M}"


# (config, layer, bits, token counts, token counts checked in full)
CASES = [
    (1, 0, (8, 8), (16,), (16,)),
    (2, 0, (8, 8), (2048,), (2048,)),
    (2, 1, (8, 8), (2048,), (2048,)),
    (2, 2, (8, 8), (2048,), (2048,)),
    (2, 3, (8, 8), (2048,), (2048,)),
    (3, 0, (6, 6), (1, 16, 128, 1024, 4096), (1, 16, 128)),
    (3, 1, (6, 6), (1, 16, 128, 1024, 4096), (1, 16, 128)),
    (3, 2, (6, 6), (1, 16, 128, 1024, 4096), (1, 16, 128)),
    (3, 3, (6, 6), (1, 16, 128, 1024, 4096), (1, 16, 128)),
    (4, 0, (8, 8), (4096,), ()),
    (4, 1, (8, 8), (4096,), ()),
    (5, 0, (8, 8), (4096,), ()),
    (5, 1, (8, 8), (4096,), ()),
    (5, 2, (8, 8), (4096,), ()),
    (5, 3, (8, 8), (4096,), ()),
    (5, 0, (6, 6), (4096,), ()),
    (5, 2, (6, 6), (4096,), ()),
]


@pytest.mark.parametrize("cfg,li,bits,Ms,full", CASES,
                         ids=[f"cfg{c}-L{l}-w{b[0]}a{b[1]}" for c, l, b, _, _ in CASES])
def test_full_size_layer(cfg, li, bits, Ms, full):
    layer, ql, o = _build_layer(cfg, li, bits)
    for M in Ms:
        _check_tokens(cfg, li, layer, ql, o, M, bits, M in full)


def test_device_timeout_status_and_recovery():
    """A bounded device wait that nothing satisfies records OT_ERR_TIMEOUT,
    the status clears once read, and the context keeps working."""
    from paper_2406_18832_gb300 import binding
    assert binding.ot_get_device_status() == binding.OT_OK
    binding.ot_selftest_wait_timeout(50_000_000)
    assert binding.ot_get_device_status() == binding.OT_ERR_TIMEOUT
    assert binding.ot_get_device_status() == binding.OT_OK
    q = torch.ones(32, 64, dtype=torch.float16, device="cuda")
    qw = torch.ones(16, 64, dtype=torch.int8, device="cuda")
    acc = torch.empty(32, 16, dtype=torch.int32, device="cuda")
    binding.ot_linear_s32(q, qw, 8, 8, acc)
    torch.cuda.synchronize()
    assert torch.all(acc == 64)
    assert binding.ot_get_device_status() == binding.OT_OK
