"""Seeded synthetic inputs shaped like the paper's OPT workloads.

This module holds no arithmetic of the method: it only draws weights, biases
and activations.  Both the CUDA path and the CPU oracle consume the tensors it
returns, so parity is judged on identical inputs.

The paper's calibration and evaluation data (Pile sentences, WikiText2/PTB/C4,
Appendix A) and its OPT checkpoints are not available; these tensors stand in
for them.  They reproduce the structure the paper describes: LayerNorm outputs
with a few fixed outlier channels that are large and asymmetric (Section 1,
Section 2.2 and Section 3.2), weights ~ N(0, 0.02).  The draws for a layer are
keyed by ``seed = 1000*config + 100*layer + stream`` with
stream 0 = weights, 1 = bias, 2 = outlier choice and parameters,
3 = calibration tokens, 4 = runtime tokens, so calibration and runtime tokens
come from the same distribution but different streams (runtime values may fall
outside the calibrated range and saturate).

Generation uses ``torch.Generator`` on the requested device; CPU and CUDA
generators give different (but each deterministic) values, and a test always
feeds the same tensors to both sides.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Layer:
    name: str
    K: int                      # input features (activation channels)
    N: int                      # output features
    outlier_frac: float = 0.005  # fraction of activation channels that are outliers
    n_outliers: int | None = None
    scale: tuple = (20.0, 80.0)  # outlier channel multiplier, uniform range
    offset: tuple = (-20.0, 20.0)  # outlier channel shift, uniform range
    post_relu: bool = False      # input follows a ReLU (non-negative, exponential tail)
    relu_out: bool = False       # ReLU fused into this layer's epilogue

    def outliers(self) -> int:
        return self.n_outliers if self.n_outliers is not None else int(round(self.outlier_frac * self.K))


@dataclass(frozen=True)
class Config:
    index: int
    name: str
    layers: tuple
    M: tuple                    # runtime token counts
    T_cal: int                  # calibration tokens per layer
    bits: tuple                 # (bits_a, bits_w) variants exercised
    extra: dict = field(default_factory=dict)


def _opt_layers(h: int, ffn: int, scale, offset, frac, fc2_relu_input=False, relu_fc1=False):
    return (
        Layer("qkv", h, 3 * h, frac, None, scale, offset),
        Layer("out", h, h, frac, None, scale, offset),
        Layer("fc1", h, ffn, frac, None, scale, offset, relu_out=relu_fc1),
        Layer("fc2", ffn, h, frac, None, scale, (0.0, 20.0) if fc2_relu_input else offset,
              post_relu=fc2_relu_input),
    )


CONFIGS = {
    # single 768x768 linear, 16 tokens, 8 outlier channels x U[20,60] + U[5,15]
    1: Config(1, "single-768", (Layer("linear", 768, 768, n_outliers=8, scale=(20.0, 60.0),
                                      offset=(5.0, 15.0)),), (16,), 64, ((8, 8),)),
    # OPT-6.7B-shaped linears, prefill of 2048 tokens, Int8, 0.5% outliers
    2: Config(2, "opt-6.7b", _opt_layers(4096, 16384, (20.0, 80.0), (-20.0, 20.0), 0.005),
              (2048,), 128 * 512, ((8, 8),)),
    # OPT-13B-shaped linears, token sweep, Int6, fc2 input after ReLU
    3: Config(3, "opt-13b", _opt_layers(5120, 20480, (20.0, 80.0), (-20.0, 20.0), 0.005,
                                        fc2_relu_input=True),
              (1, 16, 128, 1024, 4096), 128 * 512, ((6, 6),)),
    # OPT-66B-shaped fc1 / fc2, prefill of 4096 tokens, Int8, 1% outliers
    4: Config(4, "opt-66b-ffn", (Layer("fc1", 9216, 36864, 0.01, None, (30.0, 100.0), (-40.0, 40.0)),
                                 Layer("fc2", 36864, 9216, 0.01, None, (30.0, 100.0), (-40.0, 40.0))),
              (4096,), 128 * 512, ((8, 8),)),
    # OPT-30B-shaped decoder block linear path, 8 x 512 tokens, Int8 and Int6
    5: Config(5, "opt-30b-block", _opt_layers(7168, 28672, (20.0, 80.0), (-20.0, 20.0), 0.005,
                                              relu_fc1=True),
              (4096,), 128 * 512, ((8, 8), (6, 6))),
}


def seed_of(config: int, layer: int, stream: int) -> int:
    return 1000 * config + 100 * layer + stream


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def weights(cfg: int, li: int, layer: Layer, device="cpu"):
    """fp16 W[N, K] ~ N(0, 0.02) and fp16 b[N] ~ N(0, 0.01)."""
    w = torch.randn(layer.N, layer.K, generator=_gen(device, seed_of(cfg, li, 0)), device=device) * 0.02
    b = torch.randn(layer.N, generator=_gen(device, seed_of(cfg, li, 1)), device=device) * 0.01
    return w.to(torch.float16), b.to(torch.float16)


def outlier_params(cfg: int, li: int, layer: Layer, device="cpu"):
    """(channel indices, multipliers, offsets) of the fixed outlier channels."""
    g = _gen(device, seed_of(cfg, li, 2))
    idx = torch.randperm(layer.K, generator=g, device=device)[: layer.outliers()]
    n = idx.numel()
    lo, hi = layer.scale
    mult = lo + (hi - lo) * torch.rand(n, generator=g, device=device)
    olo, ohi = layer.offset
    off = olo + (ohi - olo) * torch.rand(n, generator=g, device=device)
    return idx, mult, off


def activation_chunks(cfg: int, li: int, layer: Layer, tokens: int, stream: int, device="cpu",
                      chunk: int = 8192):
    """The rows of activations(...) as consecutive fp16 blocks of `chunk`
    tokens (the same values, drawn block by block from one generator), so a
    large calibration set can be streamed without holding all of it."""
    idx, mult, off = outlier_params(cfg, li, layer, device)
    g = _gen(device, seed_of(cfg, li, stream))
    for t0 in range(0, tokens, chunk):
        t1 = min(tokens, t0 + chunk)
        if layer.post_relu:
            # zero with probability 1/2, else Exp(1)
            u = torch.rand(t1 - t0, layer.K, generator=g, device=device)
            e = -torch.log1p(-torch.rand(t1 - t0, layer.K, generator=g, device=device))
            base = torch.where(u < 0.5, torch.zeros_like(e), e)
        else:
            base = torch.randn(t1 - t0, layer.K, generator=g, device=device)
        if idx.numel():
            base[:, idx] = base[:, idx] * mult + off
        yield base.to(torch.float16)


def activations(cfg: int, li: int, layer: Layer, tokens: int, stream: int, device="cpu",
                chunk: int = 8192):
    """fp16 X[tokens, K]: N(0,1) (or ReLU'd exponential) with outlier channels.

    stream 3 = calibration tokens, stream 4 = runtime tokens.
    """
    out = torch.empty(tokens, layer.K, dtype=torch.float16, device=device)
    t0 = 0
    for blk in activation_chunks(cfg, li, layer, tokens, stream, device, chunk):
        out[t0:t0 + blk.shape[0]] = blk
        t0 += blk.shape[0]
    return out


def layer_inputs(cfg: int, li: int, tokens: int, T_cal: int | None = None, device="cpu"):
    """All tensors for one layer of a config: W, b, X_cal, X."""
    c = CONFIGS[cfg]
    layer = c.layers[li]
    w, b = weights(cfg, li, layer, device)
    xc = activations(cfg, li, layer, c.T_cal if T_cal is None else T_cal, 3, device)
    x = activations(cfg, li, layer, tokens, 4, device)
    return dict(layer=layer, W=w, b=b, X_cal=xc, X=x)
