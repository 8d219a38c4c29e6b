"""Out-of-bounds writes, checked without a memory checker: every output buffer
of every entry point that writes device memory sits between canary bytes
(0xA5), row-strided outputs carry canary columns past the row, and after the
call no byte outside the logical output may have changed.  Run at odd shapes
(M = 1, 3, 17, 200, 300; N and K = 16 x odd, and one K = 1024 prefill shape
for the CTA-pair kernel) on the release library and on the debug build, whose
kernels check their global indices (OT_DEBUG) and report a failed check
through ot_get_device_status as OT_ERR_BOUNDS.  Results are checked against
the oracle (calibration, fold, codes, linear) and, for the other entry
points, the debug build against the release library."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

DEV = "cuda"
PAD = 4096
CANARY = 0xA5


@pytest.fixture(scope="module", params=["release", "debug"])
def B(request):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2406_18832_gb300 import binding
    from paper_2406_18832_gb300 import build as _b
    if request.param == "debug":
        _b.build(debug=True)
    h = binding.select(request.param)
    assert h.ot_debug_build() == (1 if request.param == "debug" else 0)
    yield binding
    binding.select("release")


class Guarded:
    """A [rows, cols] tensor of `dtype` (row stride ld >= cols) inside a byte
    buffer whose every other byte holds the canary."""

    def __init__(self, rows, cols, dtype, ld=None):
        self.rows, self.cols, self.ld = rows, cols, ld or cols
        self.es = torch.tensor([], dtype=dtype).element_size()
        self.nbytes = rows * self.ld * self.es
        self.raw = torch.full((PAD + self.nbytes + PAD,), CANARY, dtype=torch.uint8, device=DEV)
        full = self.raw[PAD:PAD + self.nbytes].view(dtype).view(rows, self.ld)
        self.t = full[:, :cols]

    def vec(self):
        return self.t.reshape(-1) if self.rows == 1 else self.t

    def check(self, what):
        host = self.raw.cpu().numpy()
        keep = np.ones(host.size, bool)
        body = keep[PAD:PAD + self.nbytes].reshape(self.rows, self.ld * self.es)
        body[:, :self.cols * self.es] = False
        bad = np.flatnonzero(host[keep] != CANARY)
        assert bad.size == 0, f"{what}: {bad.size} canary bytes overwritten"


def _status(B):
    torch.cuda.synchronize()
    st = B.ot_get_device_status()
    assert st == B.OT_OK, B.status_string(st)


def _vec(n, dtype=torch.float32):
    return Guarded(1, n, dtype)


SHAPES = [(1, 112, 144), (3, 336, 528), (17, 1040, 2064), (200, 112, 528), (300, 528, 1024)]


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_outputs_stay_in_bounds(B, M, N, K):
    g = torch.Generator().manual_seed(M * 1000 + N + K)
    xc = torch.randn(64, K, generator=g)
    xc[:, ::37] = xc[:, ::37] * 30 + 7
    x = torch.randn(M, K, generator=g)
    x[:, ::37] = x[:, ::37] * 30 + 7
    xc, x = xc.half(), x.half()
    w = (torch.randn(N, K, generator=g) * 0.02).half()
    b = (torch.randn(N, generator=g) * 0.01).half()
    xd, xcd, wd, bd = x.to(DEV), xc.to(DEV), w.to(DEV), b.to(DEV)
    bits = 8

    # calibration and fold
    mn, mx = _vec(K), _vec(K)
    B.ot_calibrate(xcd, mn.vec(), mx.vec(), reset=True)
    z, s, r = _vec(K), _vec(K), _vec(K)
    qw = Guarded(N, K, torch.int8)
    sw, bf = _vec(N), _vec(N)
    B.ot_fold_weights(mn.vec(), mx.vec(), bits, wd, bd, bits, z.vec(), s.vec(), r.vec(), qw.t, sw.vec(), bf.vec())
    _status(B)
    for t, name in ((mn, "ch_min"), (mx, "ch_max"), (z, "z"), (s, "s"), (r, "r"), (qw, "qw"), (sw, "sw"),
                    (bf, "b'")):
        t.check(name)
    omn, omx = oracle.calibrate(xc.numpy())
    oz, os_, orr = oracle.params(omn, omx, bits)
    oqw, osw, obf = oracle.fold(w.numpy(), b.numpy(), oz, os_, bits)
    assert np.array_equal(qw.t.cpu().numpy(), oqw) and np.array_equal(bf.vec().cpu().numpy(), obf)

    # codes, both formats
    q16, q8 = Guarded(M, K, torch.float16), Guarded(M, K, torch.int8)
    B.ot_quantize_act(xd, z.vec(), r.vec(), bits, q16.t, B.OT_CODE_F16)
    B.ot_quantize_act(xd, z.vec(), r.vec(), bits, q8.t, B.OT_CODE_I8)
    _status(B)
    q16.check("fp16 codes")
    q8.check("int8 codes")
    oq = oracle.quantize(x.numpy(), oz, orr, bits)
    assert np.array_equal(q8.t.cpu().numpy(), oq)
    oacc = oracle.matmul(oq, oqw)
    oy = oracle.epilogue(oacc, osw, obf)

    # the linear: fp16 / int8 codes, with / without the stream-K workspace, strided y
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)
    for codes in (q16, q8):
        for workspace in (False, ws):
            y = Guarded(M, N, torch.float16, ld=N + 24)
            B.ot_linear(codes.t, qw.t, sw.vec(), bf.vec(), bits, bits, y.t, workspace=workspace)
            _status(B)
            y.check("y")
            assert np.array_equal(y.t.cpu().numpy().view(np.uint16), oy.view(np.uint16))
    acc = Guarded(M, N, torch.int32)
    B.ot_linear_s32(q8.t, qw.t, bits, bits, acc.t, workspace=ws)
    _status(B)
    acc.check("acc")
    assert np.array_equal(acc.t.cpu().numpy().astype(np.int64), oacc)

    # quantize + linear in one call, both forms
    for mode in (B.OT_FUSE_PDL,) + ((B.OT_FUSE_PRODUCER,) if M <= 128 else ()):
        qs, y = Guarded(M, K, torch.float16), Guarded(M, N, torch.float16, ld=N + 8)
        B.ot_linear_fused(xd, z.vec(), r.vec(), bits, qw.t, sw.vec(), bf.vec(), bits, qs.t, y.t, workspace=ws,
                          mode=mode)
        _status(B)
        qs.check("fused code scratch")
        y.check("fused y")
        assert np.array_equal(y.t.cpu().numpy().view(np.uint16), oy.view(np.uint16))

    # the next layer's codes from this epilogue (N is the next layer's K)
    qn = Guarded(M, N, torch.float16, ld=N + 16)
    zn, rn = torch.randn(N, generator=g).to(DEV), (torch.rand(N, generator=g) * 20 + 1).to(DEV)
    B.ot_linear_quantize_next(q16.t, qw.t, sw.vec(), bf.vec(), bits, bits, zn, rn, 6, qn.t, relu=True, workspace=ws)
    _status(B)
    qn.check("next-layer codes")
    on = oracle.epilogue_quantize(oacc, osw, obf, zn.cpu().numpy(), rn.cpu().numpy(), 6, True)
    assert np.array_equal(qn.t.cpu().numpy().astype(np.int64), on.astype(np.int64))


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_other_entry_points_stay_in_bounds(B, M, N, K):
    """Per-token path, asymmetric weights, LayerNorm fusion, clipping calibration."""
    g = torch.Generator().manual_seed(7 * M + N + K)
    x = (torch.randn(M, K, generator=g) * 3).half().to(DEV)
    xc = (torch.randn(257, K, generator=g) * 3).half().to(DEV)
    w = (torch.randn(N, K, generator=g) * 0.02).half().to(DEV)
    b = (torch.randn(N, generator=g) * 0.01).half().to(DEV)
    ws = torch.zeros(B.ot_linear_workspace_size(), dtype=torch.uint8, device=DEV)

    # per-token (Eq. 3)
    qt, st = Guarded(M, K, torch.float16), _vec(M)
    B.ot_quantize_tokens(x, 8, qt.t, st.vec())
    qwt, swt = Guarded(N, K, torch.int8), _vec(N)
    B.ot_quantize_weights(w, 8, qwt.t, swt.vec())
    yt = Guarded(M, N, torch.float16, ld=N + 40)
    B.ot_linear_per_token(qt.t, qwt.t, swt.vec(), st.vec(), b.float(), 8, 8, yt.t, workspace=ws)
    _status(B)
    for t, name in ((qt, "token codes"), (st, "token scales"), (qwt, "weight codes"), (swt, "sw"), (yt, "y")):
        t.check(name)
    oq, os_ = oracle.quantize_tokens(x.cpu().numpy(), 8)
    oqw, osw = oracle.quantize_weights(w.cpu().numpy(), 8)
    oy = oracle.epilogue_tokens(oracle.matmul(oq, oqw), os_, osw, b.float().cpu().numpy())
    assert np.array_equal(yt.t.cpu().numpy().view(np.uint16), oy.view(np.uint16))

    # asymmetric weights
    mn, mx = _vec(K), _vec(K)
    B.ot_calibrate(xc, mn.vec(), mx.vec(), reset=True)
    z, s, r, qwa, swa, zc, bfa = _vec(K), _vec(K), _vec(K), Guarded(N, K, torch.int8), _vec(N), \
        _vec(N, torch.int32), _vec(N)
    B.ot_fold_weights_asym(mn.vec(), mx.vec(), 8, w, b, 8, z.vec(), s.vec(), r.vec(), qwa.t, swa.vec(), zc.vec(),
                           bfa.vec())
    qa, rs = Guarded(M, K, torch.float16), _vec(M, torch.int32)
    B.ot_quantize_act_rowsum(x, z.vec(), r.vec(), 8, qa.t, rs.vec())
    ya = Guarded(M, N, torch.float16, ld=N + 8)
    B.ot_linear_asym(qa.t, qwa.t, swa.vec(), zc.vec(), rs.vec(), bfa.vec(), 8, 8, ya.t, workspace=ws)
    _status(B)
    for t, name in ((qwa, "asym codes"), (swa, "sw"), (zc, "zc"), (bfa, "b'"), (qa, "codes"), (rs, "rowsum"),
                    (ya, "y")):
        t.check(name)
    oza, osa, ora = oracle.params(*oracle.calibrate(xc.cpu().numpy()), 8)
    oqa, oswa, ozc = oracle.fold_codes_asym(w.cpu().numpy(), osa, 8)
    _, _, obfa = oracle.fold(w.cpu().numpy(), b.cpu().numpy(), oza, osa, 8)
    oqx = oracle.quantize(x.cpu().numpy(), oza, ora, 8)
    oya = oracle.epilogue_asym(oracle.matmul(oqx, oqa), oracle.rowsum(oqx), ozc, oswa, obfa)
    assert np.array_equal(ya.t.cpu().numpy().view(np.uint16), oya.view(np.uint16))

    # LayerNorm fused with the quantization
    gamma = (1 + 0.1 * torch.randn(K, generator=g)).half().to(DEV)
    beta = (0.1 * torch.randn(K, generator=g)).half().to(DEV)
    gr, br = _vec(K), _vec(K)
    B.ot_fold_layernorm(gamma, beta, z.vec(), r.vec(), gr.vec(), br.vec())
    ql, rl = Guarded(M, K, torch.int8), _vec(M, torch.int32)
    B.ot_layernorm_quantize(x, gr.vec(), br.vec(), 1e-5, 8, ql.t, B.OT_CODE_I8, rowsum=rl.vec())
    _status(B)
    for t, name in ((gr, "gamma_r"), (br, "beta_r"), (ql, "LN codes"), (rl, "LN rowsum")):
        t.check(name)
    ogr, obr = oracle.fold_layernorm(gamma.cpu().numpy(), beta.cpu().numpy(), oza, ora)
    oql, orl, _, _ = oracle.layernorm_quantize(x.cpu().numpy(), ogr, obr, 1e-5, 8)
    assert np.array_equal(ql.t.cpu().numpy(), oql) and np.array_equal(rl.vec().cpu().numpy().astype(np.int64), orl)

    # token-wise clipping calibration
    lo, hi = _vec(K), _vec(K)
    B.ot_calibrate_clipped(xc, 0.99, lo.vec(), hi.vec())
    _status(B)
    lo.check("clip lo")
    hi.check("clip hi")
    olo, ohi = oracle.calibrate_clipped(xc.cpu().numpy(), 0.99)
    assert np.array_equal(lo.vec().cpu().numpy(), olo) and np.array_equal(hi.vec().cpu().numpy(), ohi)
