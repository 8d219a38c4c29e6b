"""Helpers shared by the GPU parity tests: run one layer through the C ABI and
through the CPU oracle on the same seeded inputs."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2406_18832_gb300 import binding as B


def f16_tolerance(y_ref: np.ndarray) -> np.ndarray:
    """max(1 fp16 ulp of the reference, 1e-3 * max|y|), element-wise."""
    y = np.abs(y_ref.astype(np.float32))
    ulp = np.spacing(y.astype(np.float16)).astype(np.float32)
    return np.maximum(ulp, 1e-3 * (float(y.max()) if y.size else 0.0))


def assert_f16_close(y_gpu, y_ref, what="y"):
    y_gpu = np.asarray(y_gpu, dtype=np.float32)
    y_ref = np.asarray(y_ref, dtype=np.float32)
    err = np.abs(y_gpu - y_ref)
    tol = f16_tolerance(y_ref)
    bad = err > tol
    assert not bad.any(), f"{what}: {bad.sum()} of {bad.size} outside tolerance, worst {err.max()}"


def gpu_layer(X_cal, W, b, X, bits_a, bits_w, symmetrize=True, relu=False, out_s32=True):
    """Calibrate, fold, quantize (both code formats) and run the linear on the GPU."""
    dev = torch.device("cuda")
    K = W.shape[1]
    N = W.shape[0]
    M = X.shape[0]
    f32 = dict(dtype=torch.float32, device=dev)
    mn, mx = torch.empty(K, **f32), torch.empty(K, **f32)
    B.ot_calibrate(X_cal.to(dev), mn, mx, reset=True)
    z, s, r = (torch.empty(K, **f32) for _ in range(3))
    qw = torch.empty(N, K, dtype=torch.int8, device=dev)
    sw, bf = torch.empty(N, **f32), torch.empty(N, **f32)
    B.ot_fold_weights(mn, mx, bits_a, W.to(dev), None if b is None else b.to(dev), bits_w, z, s, r, qw, sw, bf,
                      symmetrize=symmetrize)
    Xd = X.to(dev)
    q16 = torch.empty(M, K, dtype=torch.float16, device=dev)
    q8 = torch.empty(M, K, dtype=torch.int8, device=dev)
    B.ot_quantize_act(Xd, z, r, bits_a, q16, B.OT_CODE_F16)
    B.ot_quantize_act(Xd, z, r, bits_a, q8, B.OT_CODE_I8)
    y = torch.empty(M, N, dtype=torch.float16, device=dev)
    B.ot_linear(q16, qw, sw, bf, bits_a, bits_w, y, relu=relu)
    acc = None
    if out_s32:
        acc = torch.empty(M, N, dtype=torch.int32, device=dev)
        B.ot_linear_s32(q16, qw, bits_a, bits_w, acc)
    torch.cuda.synchronize()
    assert B.ot_get_device_status() == B.OT_OK
    out = dict(mn=mn, mx=mx, z=z, s=s, r=r, qw=qw, sw=sw, bf=bf, q16=q16, q8=q8, y=y, acc=acc)
    return {k: (None if v is None else v.cpu().numpy()) for k, v in out.items()}


def oracle_layer(X_cal, W, b, X, bits_a, bits_w, symmetrize=True, relu=False, rows=None, cols=None):
    """The oracle's steps on the same inputs; rows / cols restrict the product to a sample."""
    mn, mx = oracle.calibrate(X_cal.numpy())
    z, s, r = oracle.params(mn, mx, bits_a, symmetrize)
    Wn = W.numpy()
    bn = None if b is None else b.numpy()
    if cols is not None:
        Wn = Wn[cols]
        bn = None if bn is None else bn[cols]
    qw, sw, bf = oracle.fold(Wn, bn, z, s, bits_w)
    Xn = X.numpy() if rows is None else X.numpy()[rows]
    q = oracle.quantize(Xn, z, r, bits_a)
    acc = oracle.matmul(q, qw)
    y = oracle.epilogue(acc, sw, bf, relu)
    return dict(mn=mn, mx=mx, z=z, s=s, r=r, qw=qw, sw=sw, bf=bf, q=q, acc=acc, y=y)


def compare_layer(g, o, rows=None, cols=None):
    """Bit-exact integer / parameter parity and fp16 tolerance on the output."""
    for k in ("mn", "mx", "z", "s", "r"):
        assert np.array_equal(g[k], o[k]), k
    sel_c = slice(None) if cols is None else cols
    sel_r = slice(None) if rows is None else rows
    assert np.array_equal(g["qw"][sel_c], o["qw"]), "qw"
    assert np.array_equal(g["sw"][sel_c], o["sw"]), "sw"
    assert np.array_equal(g["bf"][sel_c], o["bf"]), "b_fold"
    assert np.array_equal(g["q8"][sel_r], o["q"]), "int8 codes"
    assert np.array_equal(g["q16"][sel_r].astype(np.int64), o["q"].astype(np.int64)), "fp16 codes"
    acc_g = g["acc"][sel_r][:, sel_c] if cols is not None else g["acc"][sel_r]
    y_g = g["y"][sel_r][:, sel_c] if cols is not None else g["y"][sel_r]
    if acc_g is not None:
        assert np.array_equal(acc_g.astype(np.int64), o["acc"]), "int32 accumulators"
    assert_f16_close(y_g, o["y"])
    # the epilogue is one fp32 fma rounded to fp16 on both sides: bit-identical
    assert np.array_equal(np.asarray(y_g, np.float32), np.asarray(o["y"], np.float32)), "fp16 outputs"
