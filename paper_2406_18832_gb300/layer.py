"""QuantizedLinear: the per-channel quantized linear of OutlierTune as one
object holding the folded per-layer artefact {z, s, r, qw, sw, b'} on the GPU.

Offline (Section 3.2 "predetermined offline"; Appendix A):
    calibrate(x_cal batches) -> per-channel min / max
    fold(w, b)               -> z, s, r, qw, sw, b'   (Eq. 5, Eq. 6, Eq. 7)
Online (Eq. 6, Eq. 7):
    forward(x) = ot_linear(ot_quantize_act(x))

weights="asym" selects the paper's "Int8" weights (per-output-channel zero
points; Section 4, Appendix A): the fold also yields zero points zc, the
quantize step also yields each token's code sum, and the linear subtracts
zc_n * rowsum_m before the external scaling.

Every step is one call through the C ABI (binding.py); this class only owns
the device tensors and the stream order.
"""
from __future__ import annotations

import torch

from . import binding as B


class QuantizedLinear:
    def __init__(self, in_features: int, out_features: int, bits_a: int = 8, bits_w: int = 8,
                 symmetrize: bool = True, relu: bool = False, device="cuda", weights: str = "sym"):
        if weights not in ("sym", "asym"):
            raise ValueError("weights must be 'sym' (Int8*) or 'asym' (Int8 with zero points)")
        self.K, self.N = in_features, out_features
        self.bits_a, self.bits_w = bits_a, bits_w
        self.symmetrize, self.relu = symmetrize, relu
        self.asym = weights == "asym"
        dev = torch.device(device)
        f32 = dict(dtype=torch.float32, device=dev)
        self.ch_min = torch.empty(self.K, **f32)
        self.ch_max = torch.empty(self.K, **f32)
        self.z = torch.empty(self.K, **f32)
        self.s = torch.empty(self.K, **f32)
        self.r = torch.empty(self.K, **f32)
        self.qw = torch.empty(self.N, self.K, dtype=torch.int8, device=dev)
        self.sw = torch.empty(self.N, **f32)
        self.b_fold = torch.empty(self.N, **f32)
        self.zc = torch.empty(self.N, dtype=torch.int32, device=dev) if self.asym else None
        self._calibrated = False

    # ---- offline --------------------------------------------------------
    def calibrate(self, x_cal: torch.Tensor, stream=None):
        """Fold one batch of calibration tokens [T, K] into the running min / max."""
        B.ot_calibrate(x_cal, self.ch_min, self.ch_max, reset=not self._calibrated, stream=stream)
        self._calibrated = True
        return self

    def calibrate_clipped(self, x_cal: torch.Tensor, alpha: float = 0.999, stream=None):
        """Token-wise clipping calibration (Appendix D, for bias-free models;
        use symmetrize=False): the whole calibration set [T, K] in one call."""
        B.ot_calibrate_clipped(x_cal, alpha, self.ch_min, self.ch_max, stream=stream)
        self._calibrated = True
        return self

    def fold(self, w: torch.Tensor, b: torch.Tensor | None, stream=None):
        """Derive z, s, r from the calibration and fold them into W and b."""
        if not self._calibrated:
            raise RuntimeError("calibrate() before fold()")
        if self.asym:
            B.ot_fold_weights_asym(self.ch_min, self.ch_max, self.bits_a, w, b, self.bits_w, self.z, self.s,
                                   self.r, self.qw, self.sw, self.zc, self.b_fold, symmetrize=self.symmetrize,
                                   stream=stream)
        else:
            B.ot_fold_weights(self.ch_min, self.ch_max, self.bits_a, w, b, self.bits_w, self.z, self.s, self.r,
                              self.qw, self.sw, self.b_fold, symmetrize=self.symmetrize, stream=stream)
        return self

    def fold_layernorm(self, gamma: torch.Tensor, beta: torch.Tensor, eps: float = 1e-5, stream=None):
        """Fuse the LayerNorm in front of this linear into its quantize step
        (Section 3.2): gamma * r and (beta - z) * r, after fold()."""
        self.ln_gamma_r = torch.empty(self.K, dtype=torch.float32, device=self.z.device)
        self.ln_beta_r = torch.empty(self.K, dtype=torch.float32, device=self.z.device)
        self.ln_eps = float(eps)
        B.ot_fold_layernorm(gamma, beta, self.z, self.r, self.ln_gamma_r, self.ln_beta_r, stream=stream)
        return self

    def forward_hidden(self, h: torch.Tensor, out: torch.Tensor | None = None, stream=None):
        """y = linear(LayerNorm(h)) with the LayerNorm, symmetrization and
        quantization in one kernel (fold_layernorm() first)."""
        q = torch.empty(h.shape[0], self.K, dtype=torch.float16, device=h.device)
        rs = torch.empty(h.shape[0], dtype=torch.int32, device=h.device) if self.asym else None
        B.ot_layernorm_quantize(h, self.ln_gamma_r, self.ln_beta_r, self.ln_eps, self.bits_a, q, B.OT_CODE_F16,
                                rowsum=rs, stream=stream)
        return self.linear(q, out, stream, rowsum=rs)

    # ---- online ---------------------------------------------------------
    def quantize(self, x: torch.Tensor, out: torch.Tensor | None = None, stream=None):
        if out is None:
            out = torch.empty(x.shape[0], self.K, dtype=torch.float16, device=x.device)
        B.ot_quantize_act(x, self.z, self.r, self.bits_a, out, B.OT_CODE_F16, stream=stream)
        return out

    def quantize_with_rowsum(self, x: torch.Tensor, out: torch.Tensor | None = None,
                             rowsum: torch.Tensor | None = None, stream=None):
        """Codes and each token's code sum (int32 [M]), for the asymmetric weights."""
        if out is None:
            out = torch.empty(x.shape[0], self.K, dtype=torch.float16, device=x.device)
        if rowsum is None:
            rowsum = torch.empty(x.shape[0], dtype=torch.int32, device=x.device)
        B.ot_quantize_act_rowsum(x, self.z, self.r, self.bits_a, out, rowsum, B.OT_CODE_F16, stream=stream)
        return out, rowsum

    def linear(self, q: torch.Tensor, out: torch.Tensor | None = None, stream=None,
               rowsum: torch.Tensor | None = None):
        if out is None:
            out = torch.empty(q.shape[0], self.N, dtype=torch.float16, device=q.device)
        if self.asym:
            if rowsum is None:
                raise ValueError("asymmetric weights need the codes' row sums (quantize_with_rowsum)")
            B.ot_linear_asym(q, self.qw, self.sw, self.zc, rowsum, self.b_fold, self.bits_a, self.bits_w, out,
                             relu=self.relu, stream=stream)
        else:
            B.ot_linear(q, self.qw, self.sw, self.b_fold, self.bits_a, self.bits_w, out, relu=self.relu,
                        stream=stream)
        return out

    def linear_quantize_next(self, q: torch.Tensor, nxt: "QuantizedLinear", out: torch.Tensor | None = None,
                             stream=None):
        """This layer's linear with the next layer's activation quantization in
        its epilogue (Section 3.2): returns nxt's fp16 codes [M, N], the q that
        nxt.linear takes, without this layer's fp16 output."""
        if self.asym:
            raise ValueError("the chained epilogue takes symmetric weights")
        if nxt.K != self.N:
            raise ValueError("the next layer's in_features must equal this layer's out_features")
        if out is None:
            out = torch.empty(q.shape[0], self.N, dtype=torch.float16, device=q.device)
        B.ot_linear_quantize_next(q, self.qw, self.sw, self.b_fold, self.bits_a, self.bits_w, nxt.z, nxt.r,
                                  nxt.bits_a, out, relu=self.relu, stream=stream)
        return out

    def forward(self, x: torch.Tensor, q_buf: torch.Tensor | None = None, out: torch.Tensor | None = None,
                stream=None):
        if self.asym:
            q, rs = self.quantize_with_rowsum(x, q_buf, stream=stream)
            return self.linear(q, out, stream, rowsum=rs)
        return self.linear(self.quantize(x, q_buf, stream), out, stream)

    __call__ = forward

    def state_dict(self):
        """The per-layer artefact, as plain tensors (saved with torch.save)."""
        keys = ("ch_min", "ch_max", "z", "s", "r", "qw", "sw", "b_fold") + (("zc",) if self.asym else ())
        return {k: getattr(self, k) for k in keys}

    def load_state_dict(self, sd):
        for k, v in sd.items():
            getattr(self, k).copy_(v)
        self._calibrated = True
        return self

    def weight_bytes(self) -> int:
        return self.qw.numel() + 4 * (self.sw.numel() + self.b_fold.numel() + (self.N if self.asym else 0))


class QuantizedBlockLinears:
    """The linear path of one OPT-style decoder block, every layer per-channel
    quantized with its own calibration (the paper applies the method to the
    linears after LayerNorm and keeps residual / LayerNorm / attention in
    fp16; those are not part of this path):

        qkv = QKV(x);  v = qkv[:, 2h:3h]   (stand-in for attention: its V slice)
        o   = out(v);  f = ReLU(fc1(o));   y = fc2(f)

    calibrate() runs the calibration tokens through the already-folded
    layers, so each layer is calibrated on the activations it receives.
    """

    def __init__(self, hidden: int, ffn: int, bits_a: int = 8, bits_w: int = 8, device="cuda"):
        self.h, self.ffn = hidden, ffn
        mk = lambda K, N, relu=False: QuantizedLinear(K, N, bits_a, bits_w, relu=relu, device=device)
        self.qkv = mk(hidden, 3 * hidden)
        self.out = mk(hidden, hidden)
        self.fc1 = mk(hidden, ffn, relu=True)
        self.fc2 = mk(ffn, hidden)
        self.layers = (self.qkv, self.out, self.fc1, self.fc2)

    def calibrate(self, x_cal: torch.Tensor, weights, batch: int = 8192, stream=None):
        """weights: [(w, b)] for qkv, out, fc1, fc2 (fp16, [N, K] and [N])."""
        acts = x_cal
        for i, (ql, (w, b)) in enumerate(zip(self.layers, weights)):
            for t0 in range(0, acts.shape[0], batch):
                ql.calibrate(acts[t0:t0 + batch], stream=stream)
            ql.fold(w, b, stream=stream)
            if i + 1 < len(self.layers):
                nxt = torch.empty(acts.shape[0], ql.N, dtype=torch.float16, device=acts.device)
                for t0 in range(0, acts.shape[0], batch):
                    ql.forward(acts[t0:t0 + batch], out=nxt[t0:t0 + batch], stream=stream)
                acts = nxt[:, 2 * self.h:] if ql is self.qkv else nxt
        return self

    def forward(self, x: torch.Tensor, stream=None, fused: bool = False):
        """All intermediate outputs: qkv, o, f, y (fp16).  fused=True chains
        fc1 into fc2 through codes: fc1's epilogue (ReLU) writes fc2's
        activation codes qf in place of f, so f never reaches HBM."""
        qkv = self.qkv(x, stream=stream)
        o = self.out(qkv[:, 2 * self.h:], stream=stream)
        if fused:
            qf = self.fc1.linear_quantize_next(self.fc1.quantize(o, stream=stream), self.fc2, stream=stream)
            return dict(qkv=qkv, o=o, qf=qf, y=self.fc2.linear(qf, stream=stream))
        f = self.fc1(o, stream=stream)
        y = self.fc2(f, stream=stream)
        return dict(qkv=qkv, o=o, f=f, y=y)

    def weight_bytes(self) -> int:
        return sum(ql.weight_bytes() for ql in self.layers)
