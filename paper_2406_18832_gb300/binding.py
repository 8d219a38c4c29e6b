"""Thin Python binding of the C ABI in include/outliertune.h.

Argument marshalling only: every function takes CUDA torch tensors, checks
that they live on the GPU with the dtype and layout the C function expects,
and passes raw pointers, sizes and the current CUDA stream.  All arithmetic
runs in the CUDA library; there is no CPU fallback: if the library is not
built, or a tensor is not on a CUDA device, the call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

OT_OK, OT_ERR_INVALID_ARG, OT_ERR_UNSUPPORTED, OT_ERR_CUDA, OT_ERR_TIMEOUT, OT_ERR_BOUNDS = range(6)
OT_CODE_I8, OT_CODE_F16 = 0, 1
OT_FUSE_AUTO, OT_FUSE_PRODUCER, OT_FUSE_PDL = 0, 1, 2

_lock = threading.Lock()
_handle = None          # the library the functions below call
_handles = {}           # loaded libraries by variant ("release", "debug")

_P, _I64, _I, _F = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float
_SIGNATURES = {
    "ot_status_string": ([_I], ctypes.c_char_p),
    "ot_version": ([], _I),
    "ot_debug_build": ([], _I),
    "ot_calibrate": ([_P, _I64, _I64, _I64, _P, _P, _I, _P], _I),
    "ot_derive_params": ([_P, _P, _I64, _I, _I, _P, _P, _P, _P], _I),
    "ot_fold_weights": ([_P, _P, _I, _I, _P, _P, _I64, _I64, _I, _P, _P, _P, _P, _P, _P, _P], _I),
    "ot_quantize_act": ([_P, _I64, _I64, _I64, _P, _P, _I, _P, _I, _P], _I),
    "ot_linear": ([_P, _I, _I64, _I64, _P, _P, _P, _I64, _I, _I, _P, _I64, _I, _P, ctypes.c_size_t, _P], _I),
    "ot_linear_s32": ([_P, _I, _I64, _I64, _P, _I64, _I, _I, _P, _P, ctypes.c_size_t, _P], _I),
    "ot_linear_workspace_size": ([_P], _I),
    "ot_linear_noalloc": ([_P, _I64, _I64, _P, _P, _P, _I64, _I, _I, _P, _I64, _I, _P], _I),
    "ot_quantize_tokens": ([_P, _I64, _I64, _I64, _I, _P, _I, _P, _P], _I),
    "ot_quantize_weights": ([_P, _I64, _I64, _I, _P, _P, _P], _I),
    "ot_linear_per_token": ([_P, _I64, _I64, _P, _P, _P, _P, _I64, _I, _I, _P, _I64, _I, _P, ctypes.c_size_t, _P],
                            _I),
    "ot_fold_weights_asym": ([_P, _P, _I, _I, _P, _P, _I64, _I64, _I, _P, _P, _P, _P, _P, _P, _P, _P], _I),
    "ot_quantize_act_rowsum": ([_P, _I64, _I64, _I64, _P, _P, _I, _P, _I, _P, _P], _I),
    "ot_linear_asym": ([_P, _I64, _I64, _P, _P, _P, _P, _P, _I64, _I, _I, _P, _I64, _I, _P, ctypes.c_size_t, _P],
                       _I),
    "ot_fold_layernorm": ([_P, _P, _P, _P, _I64, _P, _P, _P], _I),
    "ot_layernorm_quantize": ([_P, _I64, _I64, _I64, _P, _P, _F, _I, _P, _I, _P, _P], _I),
    "ot_calibrate_clipped": ([_P, _I64, _I64, _I64, ctypes.c_double, _P, _P, _P], _I),
    "ot_linear_quantize_next": ([_P, _I64, _I64, _P, _P, _P, _I64, _I, _I, _I, _P, _P, _I, _P, _I64, _P,
                                 ctypes.c_size_t, _P], _I),
    "ot_linear_fused": ([_P, _I64, _I64, _I64, _P, _P, _I, _P, _P, _P, _I64, _I, _P, _P, _I64, _I, _I, _P,
                         ctypes.c_size_t, _P], _I),
    "ot_get_device_status": ([_P], _I),
    "ot_selftest_wait_timeout": ([_I64, _P], _I),
}


class OTError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)}")


def library_path() -> str:
    return _build.LIB_PATH


def _open(variant: str) -> ctypes.CDLL:
    lib = _handles.get(variant)
    if lib is None:
        path = _build.LIB_PATH_DEBUG if variant == "debug" else _build.LIB_PATH
        if not os.path.exists(path):
            raise RuntimeError(f"CUDA library not built: {path} is missing "
                               "(run __graft_entry__.build() or python -m paper_2406_18832_gb300.build)")
        lib = ctypes.CDLL(path)
        for name, (args, res) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _handles[variant] = lib
    return lib


def load() -> ctypes.CDLL:
    """The library the functions of this module call: lib/libot_gb300.so
    (built by paper_2406_18832_gb300.build) unless select() chose another."""
    global _handle
    with _lock:
        if _handle is None:
            _handle = _open("release")
    return _handle


def select(variant: str = "release") -> ctypes.CDLL:
    """Route this module's calls to the release library or to the debug build
    (lib/libot_gb300_debug.so: kernels check their indices, OT_DEBUG)."""
    global _handle
    if variant not in ("release", "debug"):
        raise ValueError("variant must be 'release' or 'debug'")
    with _lock:
        _handle = _open(variant)
    return _handle


def status_string(status: int) -> str:
    return load().ot_status_string(int(status)).decode()


def version() -> int:
    return load().ot_version()


def _check(status: int, where: str):
    if status != OT_OK:
        raise OTError(status, where)


def _dev(t: torch.Tensor, name: str, dtype=None) -> int:
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (the library takes device pointers)")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def _dense(t: torch.Tensor, name: str):
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _rows(t: torch.Tensor, name: str):
    """(rows, cols, row stride) of a 2-D tensor with unit column stride."""
    if t.dim() != 2 or (t.shape[1] > 1 and t.stride(1) != 1):
        raise ValueError(f"{name} must be 2-D with unit stride along its last dimension")
    return t.shape[0], t.shape[1], t.stride(0) if t.shape[0] > 1 else t.shape[1]


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def ot_calibrate(x: torch.Tensor, ch_min: torch.Tensor, ch_max: torch.Tensor, reset: bool = True, stream=None):
    """Per-channel running min / max of fp16 X[T, K] into fp32 ch_min, ch_max [K]."""
    T, K, ldx = _rows(x, "x")
    px = _dev(x, "x", torch.float16)
    _check(load().ot_calibrate(px, T, K, ldx, _dev(ch_min, "ch_min", torch.float32),
                               _dev(ch_max, "ch_max", torch.float32), 1 if reset else 0, _stream(stream)),
           "ot_calibrate")


def ot_calibrate_clipped(x: torch.Tensor, alpha: float, ch_lo: torch.Tensor, ch_hi: torch.Tensor, stream=None):
    """Token-wise clipped per-channel range of fp16 X_cal [T, K] at quantile alpha (order statistics)."""
    T, K, ldx = _rows(x, "x")
    _check(load().ot_calibrate_clipped(_dev(x, "x", torch.float16), T, K, ldx, float(alpha),
                                       _dev(ch_lo, "ch_lo", torch.float32), _dev(ch_hi, "ch_hi", torch.float32),
                                       _stream(stream)),
           "ot_calibrate_clipped")


def ot_derive_params(ch_min, ch_max, bits_a: int, z, s, r, symmetrize: bool = True, stream=None):
    K = ch_min.numel()
    _check(load().ot_derive_params(_dev(ch_min, "ch_min", torch.float32), _dev(ch_max, "ch_max", torch.float32), K,
                                   bits_a, 1 if symmetrize else 0, _dev(z, "z", torch.float32),
                                   _dev(s, "s", torch.float32), _dev(r, "r", torch.float32), _stream(stream)),
           "ot_derive_params")


def ot_fold_weights(ch_min, ch_max, bits_a: int, w, b, bits_w: int, z, s, r, qw, sw, b_fold,
                    symmetrize: bool = True, stream=None):
    _dense(w, "w")
    N, K = w.shape
    pb = None if b is None else _dev(b, "b", torch.float16)
    _check(load().ot_fold_weights(_dev(ch_min, "ch_min", torch.float32), _dev(ch_max, "ch_max", torch.float32),
                                  bits_a, 1 if symmetrize else 0, _dev(w, "w", torch.float16), pb, N, K, bits_w,
                                  _dev(z, "z", torch.float32), _dev(s, "s", torch.float32),
                                  _dev(r, "r", torch.float32), _dev(qw, "qw", torch.int8),
                                  _dev(sw, "sw", torch.float32), _dev(b_fold, "b_fold", torch.float32),
                                  _stream(stream)),
           "ot_fold_weights")


def ot_quantize_act(x, z, r, bits_a: int, q, q_format: int = OT_CODE_F16, stream=None):
    M, K, ldx = _rows(x, "x")
    _dense(q, "q")
    want = torch.float16 if q_format == OT_CODE_F16 else torch.int8
    _check(load().ot_quantize_act(_dev(x, "x", torch.float16), M, K, ldx, _dev(z, "z", torch.float32),
                                  _dev(r, "r", torch.float32), bits_a, _dev(q, "q", want), q_format,
                                  _stream(stream)),
           "ot_quantize_act")


def ot_fold_weights_asym(ch_min, ch_max, bits_a: int, w, b, bits_w: int, z, s, r, qw, sw, zc, b_fold,
                         symmetrize: bool = True, stream=None):
    """ot_fold_weights with asymmetric per-output-channel codes (the paper's "Int8"):
    qw int8 [N, K] stored as u - 2^(b-1), zero points zc int32 [N]."""
    _dense(w, "w")
    N, K = w.shape
    pb = None if b is None else _dev(b, "b", torch.float16)
    _check(load().ot_fold_weights_asym(_dev(ch_min, "ch_min", torch.float32),
                                       _dev(ch_max, "ch_max", torch.float32), bits_a, 1 if symmetrize else 0,
                                       _dev(w, "w", torch.float16), pb, N, K, bits_w, _dev(z, "z", torch.float32),
                                       _dev(s, "s", torch.float32), _dev(r, "r", torch.float32),
                                       _dev(qw, "qw", torch.int8), _dev(sw, "sw", torch.float32),
                                       _dev(zc, "zc", torch.int32), _dev(b_fold, "b_fold", torch.float32),
                                       _stream(stream)),
           "ot_fold_weights_asym")


def ot_quantize_act_rowsum(x, z, r, bits_a: int, q, rowsum, q_format: int = OT_CODE_F16, stream=None):
    """ot_quantize_act plus rowsum[m] = sum_k q[m, k] (int32 [M])."""
    M, K, ldx = _rows(x, "x")
    _dense(q, "q")
    want = torch.float16 if q_format == OT_CODE_F16 else torch.int8
    _check(load().ot_quantize_act_rowsum(_dev(x, "x", torch.float16), M, K, ldx, _dev(z, "z", torch.float32),
                                         _dev(r, "r", torch.float32), bits_a, _dev(q, "q", want), q_format,
                                         _dev(rowsum, "rowsum", torch.int32), _stream(stream)),
           "ot_quantize_act_rowsum")


def ot_linear_asym(q, qw, sw, zc, rowsum, b_fold, bits_a: int, bits_w: int, y, relu: bool = False,
                   workspace=None, stream=None):
    """y = fp16(fma((float)(acc - zc_n rowsum_m), sw_n, b'_n)) with asymmetric weight codes."""
    _dense(q, "q")
    _dense(qw, "qw")
    M, K = q.shape
    N = qw.shape[0]
    ym, yn, ldy = _rows(y, "y")
    if ym != M or yn != N:
        raise ValueError("y must be [M, N]")
    wp, wb = _ws_args(workspace, q.device, stream)
    _check(load().ot_linear_asym(_dev(q, "q", torch.float16), M, K, _dev(qw, "qw", torch.int8),
                                 _dev(sw, "sw", torch.float32), _dev(zc, "zc", torch.int32),
                                 _dev(rowsum, "rowsum", torch.int32), _dev(b_fold, "b_fold", torch.float32), N,
                                 bits_a, bits_w, _dev(y, "y", torch.float16), ldy, 1 if relu else 0, wp, wb,
                                 _stream(stream)),
           "ot_linear_asym")


def ot_fold_layernorm(gamma, beta, z, r, gamma_r, beta_r, stream=None):
    """gamma_r = gamma * r, beta_r = (beta - z) * r (fp32 [K]) from the LayerNorm's fp16 gamma, beta."""
    K = gamma.numel()
    _check(load().ot_fold_layernorm(_dev(gamma, "gamma", torch.float16), _dev(beta, "beta", torch.float16),
                                    _dev(z, "z", torch.float32), _dev(r, "r", torch.float32), K,
                                    _dev(gamma_r, "gamma_r", torch.float32), _dev(beta_r, "beta_r", torch.float32),
                                    _stream(stream)),
           "ot_fold_layernorm")


def ot_layernorm_quantize(h, gamma_r, beta_r, eps: float, bits_a: int, q, q_format: int = OT_CODE_F16,
                          rowsum=None, stream=None):
    """Codes of the symmetrized LayerNorm output of fp16 h [M, K] (optionally their row sums)."""
    M, K, ldh = _rows(h, "h")
    _dense(q, "q")
    want = torch.float16 if q_format == OT_CODE_F16 else torch.int8
    prs = None if rowsum is None else _dev(rowsum, "rowsum", torch.int32)
    _check(load().ot_layernorm_quantize(_dev(h, "h", torch.float16), M, K, ldh, _dev(gamma_r, "gamma_r", torch.float32),
                                        _dev(beta_r, "beta_r", torch.float32), float(eps), bits_a,
                                        _dev(q, "q", want), q_format, prs, _stream(stream)),
           "ot_layernorm_quantize")


def ot_linear_fused(x, z, r, bits_a: int, qw, sw, b_fold, bits_w: int, q, y, relu: bool = False, workspace=None,
                    stream=None, mode: int = OT_FUSE_AUTO):
    """Quantize x and run the linear into y [M, N] in one call; q is fp16 scratch [M, K]; mode is an
    ot_fuse_mode (OT_FUSE_PRODUCER: quantized inside the linear, up to 128 tokens)."""
    M, K, ldx = _rows(x, "x")
    _dense(q, "q")
    _dense(qw, "qw")
    N = qw.shape[0]
    if tuple(q.shape) != (M, K):
        raise ValueError("q must be [M, K]")
    ym, yn, ldy = _rows(y, "y")
    if ym != M or yn != N:
        raise ValueError("y must be [M, N]")
    wp, wb = _ws_args(workspace, x.device, stream)
    _check(load().ot_linear_fused(_dev(x, "x", torch.float16), M, K, ldx, _dev(z, "z", torch.float32),
                                  _dev(r, "r", torch.float32), bits_a, _dev(qw, "qw", torch.int8),
                                  _dev(sw, "sw", torch.float32), _dev(b_fold, "b_fold", torch.float32), N, bits_w,
                                  _dev(q, "q", torch.float16), _dev(y, "y", torch.float16), ldy, 1 if relu else 0,
                                  mode, wp, wb, _stream(stream)), "ot_linear_fused")


def ot_linear_quantize_next(q, qw, sw, b_fold, bits_a: int, bits_w: int, z_next, r_next, bits_next: int, q_next,
                            relu: bool = False, workspace=None, stream=None):
    """The linear whose epilogue writes the next layer's fp16 codes q_next [M, N] (fc1 -> ReLU -> fc2)."""
    _dense(q, "q")
    _dense(qw, "qw")
    M, K = q.shape
    N = qw.shape[0]
    qm, qn, ldq = _rows(q_next, "q_next")
    if qm != M or qn != N:
        raise ValueError("q_next must be [M, N]")
    wp, wb = _ws_args(workspace, q.device, stream)
    _check(load().ot_linear_quantize_next(_dev(q, "q", torch.float16), M, K, _dev(qw, "qw", torch.int8),
                                          _dev(sw, "sw", torch.float32), _dev(b_fold, "b_fold", torch.float32), N,
                                          bits_a, bits_w, 1 if relu else 0, _dev(z_next, "z_next", torch.float32),
                                          _dev(r_next, "r_next", torch.float32), bits_next,
                                          _dev(q_next, "q_next", torch.float16), ldq, wp, wb, _stream(stream)),
           "ot_linear_quantize_next")


def ot_linear_workspace_size() -> int:
    """Bytes of stream-K scratch for prefill-sized linears on the current device."""
    n = ctypes.c_size_t(0)
    _check(load().ot_linear_workspace_size(ctypes.byref(n)), "ot_linear_workspace_size")
    return int(n.value)


_workspaces = {}


def default_workspace(device=None, stream=None) -> torch.Tensor:
    """A zero-filled scratch tensor for ot_linear, one per (device, stream): the
    library allocates nothing itself, and calls that overlap on the GPU must not
    share a workspace, so each stream gets its own."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    key = (dev.index, _stream(stream))
    ws = _workspaces.get(key)
    if ws is None:
        with torch.cuda.device(dev):
            ws = torch.zeros(ot_linear_workspace_size(), dtype=torch.uint8, device=dev)
        _workspaces[key] = ws
    return ws


def _ws_args(workspace, device, stream):
    """(pointer, bytes) for the workspace argument: None picks the per-stream
    default, False passes none (whole tiles dealt out)."""
    if workspace is False:
        return None, 0
    if workspace is None:
        workspace = default_workspace(device, stream)
    return _dev(workspace, "workspace"), workspace.numel() * workspace.element_size()


def _codes(q):
    """(pointer, ot_code_format) of an activation-code tensor: int8 or fp16 codes."""
    if q.dtype == torch.int8:
        return _dev(q, "q", torch.int8), OT_CODE_I8
    return _dev(q, "q", torch.float16), OT_CODE_F16


def ot_linear(q, qw, sw, b_fold, bits_a: int, bits_w: int, y, relu: bool = False, workspace=None, stream=None):
    """y = fp16(fma(sum_k q qw, sw, b')); q holds int8 or fp16 codes (its dtype picks the format)."""
    _dense(q, "q")
    _dense(qw, "qw")
    M, K = q.shape
    N = qw.shape[0]
    ym, yn, ldy = _rows(y, "y")
    if ym != M or yn != N:
        raise ValueError("y must be [M, N]")
    pq, fmt = _codes(q)
    wp, wb = _ws_args(workspace, q.device, stream)
    _check(load().ot_linear(pq, fmt, M, K, _dev(qw, "qw", torch.int8), _dev(sw, "sw", torch.float32),
                            _dev(b_fold, "b_fold", torch.float32), N, bits_a, bits_w,
                            _dev(y, "y", torch.float16), ldy, 1 if relu else 0, wp, wb, _stream(stream)),
           "ot_linear")


def ot_quantize_tokens(x, bits_a: int, q, s_tok, q_format: int = OT_CODE_F16, stream=None):
    """Per-token dynamic codes and scales of fp16 X[M, K] (Eq. 3)."""
    M, K, ldx = _rows(x, "x")
    _dense(q, "q")
    want = torch.float16 if q_format == OT_CODE_F16 else torch.int8
    _check(load().ot_quantize_tokens(_dev(x, "x", torch.float16), M, K, ldx, bits_a, _dev(q, "q", want), q_format,
                                     _dev(s_tok, "s_tok", torch.float32), _stream(stream)),
           "ot_quantize_tokens")


def ot_quantize_weights(w, bits_w: int, qw, sw, stream=None):
    """Per-output-channel weight codes without activation scales (Eq. 3's W~)."""
    _dense(w, "w")
    N, K = w.shape
    _check(load().ot_quantize_weights(_dev(w, "w", torch.float16), N, K, bits_w, _dev(qw, "qw", torch.int8),
                                      _dev(sw, "sw", torch.float32), _stream(stream)),
           "ot_quantize_weights")


def ot_linear_per_token(q, qw, sw, s_tok, bias, bits_a: int, bits_w: int, y, relu: bool = False, workspace=None,
                        stream=None):
    _dense(q, "q")
    _dense(qw, "qw")
    M, K = q.shape
    N = qw.shape[0]
    ym, yn, ldy = _rows(y, "y")
    if ym != M or yn != N:
        raise ValueError("y must be [M, N]")
    pq = _dev(q, "q", torch.float16)
    wp, wb = _ws_args(workspace, q.device, stream)
    _check(load().ot_linear_per_token(pq, M, K, _dev(qw, "qw", torch.int8), _dev(sw, "sw", torch.float32),
                                      _dev(s_tok, "s_tok", torch.float32), _dev(bias, "bias", torch.float32), N,
                                      bits_a, bits_w, _dev(y, "y", torch.float16), ldy, 1 if relu else 0, wp, wb,
                                      _stream(stream)),
           "ot_linear_per_token")


def ot_linear_noalloc(q, qw, sw, b_fold, bits_a: int, bits_w: int, y, relu: bool = False, stream=None):
    """ot_linear through the entry point that allocates nothing (its scratch is
    a fixed array inside the library, shared by every call)."""
    _dense(q, "q")
    _dense(qw, "qw")
    M, K = q.shape
    N = qw.shape[0]
    ym, yn, ldy = _rows(y, "y")
    if ym != M or yn != N:
        raise ValueError("y must be [M, N]")
    _check(load().ot_linear_noalloc(_dev(q, "q", torch.float16), M, K, _dev(qw, "qw", torch.int8),
                                    _dev(sw, "sw", torch.float32), _dev(b_fold, "b_fold", torch.float32), N,
                                    bits_a, bits_w, _dev(y, "y", torch.float16), ldy, 1 if relu else 0,
                                    _stream(stream)),
           "ot_linear_noalloc")


def ot_linear_s32(q, qw, bits_a: int, bits_w: int, acc, workspace=None, stream=None):
    _dense(q, "q")
    _dense(qw, "qw")
    _dense(acc, "acc")
    M, K = q.shape
    N = qw.shape[0]
    pq, fmt = _codes(q)
    wp, wb = _ws_args(workspace, q.device, stream)
    _check(load().ot_linear_s32(pq, fmt, M, K, _dev(qw, "qw", torch.int8), N, bits_a, bits_w,
                                _dev(acc, "acc", torch.int32), wp, wb, _stream(stream)),
           "ot_linear_s32")


def ot_get_device_status(stream=None) -> int:
    return load().ot_get_device_status(_stream(stream))


def ot_selftest_wait_timeout(limit_ns: int = 50_000_000, stream=None):
    _check(load().ot_selftest_wait_timeout(int(limit_ns), _stream(stream)), "ot_selftest_wait_timeout")
