"""QuantizedLinear: the per-channel quantized linear of OutlierTune as one
object holding the folded per-layer artefact {z, s, r, qw, sw, b'} on the GPU.

Offline (Section 3.2 "predetermined offline"; Appendix A):
    calibrate(x_cal batches) -> per-channel min / max
    fold(w, b)               -> z, s, r, qw, sw, b'   (Eq. 5, Eq. 6, Eq. 7)
Online (Eq. 6, Eq. 7):
    forward(x) = ot_linear(ot_quantize_act(x))

Every step is one call through the C ABI (binding.py); this class only owns
the device tensors and the stream order.
"""
from __future__ import annotations

import torch

from . import binding as B


class QuantizedLinear:
    def __init__(self, in_features: int, out_features: int, bits_a: int = 8, bits_w: int = 8,
                 symmetrize: bool = True, relu: bool = False, device="cuda"):
        self.K, self.N = in_features, out_features
        self.bits_a, self.bits_w = bits_a, bits_w
        self.symmetrize, self.relu = symmetrize, relu
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
        self._calibrated = False

    # ---- offline --------------------------------------------------------
    def calibrate(self, x_cal: torch.Tensor, stream=None):
        """Fold one batch of calibration tokens [T, K] into the running min / max."""
        B.ot_calibrate(x_cal, self.ch_min, self.ch_max, reset=not self._calibrated, stream=stream)
        self._calibrated = True
        return self

    def fold(self, w: torch.Tensor, b: torch.Tensor | None, stream=None):
        """Derive z, s, r from the calibration and fold them into W and b."""
        if not self._calibrated:
            raise RuntimeError("calibrate() before fold()")
        B.ot_fold_weights(self.ch_min, self.ch_max, self.bits_a, w, b, self.bits_w, self.z, self.s, self.r,
                          self.qw, self.sw, self.b_fold, symmetrize=self.symmetrize, stream=stream)
        return self

    # ---- online ---------------------------------------------------------
    def quantize(self, x: torch.Tensor, out: torch.Tensor | None = None, stream=None):
        if out is None:
            out = torch.empty(x.shape[0], self.K, dtype=torch.float16, device=x.device)
        B.ot_quantize_act(x, self.z, self.r, self.bits_a, out, B.OT_CODE_F16, stream=stream)
        return out

    def linear(self, q: torch.Tensor, out: torch.Tensor | None = None, stream=None):
        if out is None:
            out = torch.empty(q.shape[0], self.N, dtype=torch.float16, device=q.device)
        B.ot_linear(q, self.qw, self.sw, self.b_fold, self.bits_a, self.bits_w, out, relu=self.relu,
                    stream=stream)
        return out

    def forward(self, x: torch.Tensor, q_buf: torch.Tensor | None = None, out: torch.Tensor | None = None,
                stream=None):
        return self.linear(self.quantize(x, q_buf, stream), out, stream)

    __call__ = forward

    def state_dict(self):
        """The per-layer artefact, as plain tensors (saved with torch.save)."""
        return {k: getattr(self, k) for k in ("ch_min", "ch_max", "z", "s", "r", "qw", "sw", "b_fold")}

    def load_state_dict(self, sd):
        for k, v in sd.items():
            getattr(self, k).copy_(v)
        self._calibrated = True
        return self

    def weight_bytes(self) -> int:
        return self.qw.numel() + 4 * (self.sw.numel() + self.b_fold.numel())
