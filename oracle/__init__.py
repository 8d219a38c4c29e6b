"""CPU oracle of the OutlierTune per-channel quantized linear (arXiv 2406.18832).

TEST INFRASTRUCTURE ONLY: imported by the tests, by ``__graft_entry__.smoke()``
and by the ``cpu_baseline`` leg of ``bench.py``; never by the product package.
It shares no code with the CUDA library.  The arithmetic lives in plain C
(``ot_oracle.c``, compiled here with gcc, no FMA contraction, no fast-math);
this module only builds it and marshals numpy arrays.

Functions follow the paper's steps in order:
  calibrate  - per-channel min/max (Appendix A; Section 3.2)
  params     - z = (max+min)/2 and the static scale s (Section 3.2; Eq. 1)
  fold       - W_s = W (.) s (Eq. 5), per-output-channel codes (Eq. 6),
               b' = b + z W^T (Eq. 7)
  quantize   - round((X - z) / s) (Eq. 6, Eq. 7)
  matmul     - sum_k q[m,k] qw[n,k] in int64 (Eq. 6)
  epilogue   - fp16(fma((float)acc, sw, b')) (Eq. 6, Eq. 7)
and the per-token path of Eq. 3 (the paper's out / fc2 linears):
  quantize_tokens   - dynamic per-token scale s_m = max|x[m,:]| / qmax and codes
  quantize_weights  - per-output-channel codes of W without activation scales
  epilogue_tokens   - fp16(fma((float)acc, s_m * sw_n, b_n))
and the asymmetric weights ("Int8": per-output-channel zero points, Eq. 1):
  fold_codes_asym   - codes of W_s over [min(0, min), max(0, max)] with a zero point
  rowsum            - sum_k q[m,k] (exact)
  epilogue_asym     - fp16(fma((float)(acc - zc_n rs_m), sw_n, b'_n))
and the LayerNorm fused with the symmetrization and quantization (Section 3.2):
  fold_layernorm       - gamma * r and (beta - z) * r
  layernorm_quantize   - exact row statistics, codes of LN(h) - z scaled by r
and the token-wise clipping calibration of bias-free models (Appendix D):
  calibrate_clipped    - per-channel order statistics at quantile alpha
and the epilogue that writes the next linear's codes (fc1 -> ReLU -> fc2):
  epilogue_quantize    - round((fma(acc, sw, b') [ReLU] - z') * r')
Threaded drivers (calibrate_mt, fold_mt, quantize_mt, matmul_mt,
epilogue_mt) run the same C functions on disjoint row or channel ranges in
parallel host threads, for full-size parity checks and the timed CPU
baseline; their results are identical to the single-threaded calls.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ot_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libot_oracle.so")
_CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ot_oracle.c into oracle/_build/libot_oracle.so (gcc)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", *_CFLAGS, _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            I64 = ctypes.c_int64
            I = ctypes.c_int
            lib.ot_half_to_float.argtypes = [ctypes.c_uint16]
            lib.ot_half_to_float.restype = ctypes.c_float
            lib.ot_double_to_half.argtypes = [ctypes.c_double]
            lib.ot_double_to_half.restype = ctypes.c_uint16
            lib.oracle_calibrate.argtypes = [P, I64, I64, I64, P, P, I]
            lib.oracle_params.argtypes = [P, P, I64, I, I, P, P, P]
            lib.oracle_fold.argtypes = [P, P, I64, I64, P, P, I, P, P, P]
            lib.oracle_quantize.argtypes = [P, I64, I64, I64, P, P, I, P]
            lib.oracle_matmul.argtypes = [P, P, I64, I64, I64, P]
            lib.oracle_epilogue.argtypes = [P, I64, I64, P, P, I, P]
            lib.oracle_quantize_tokens.argtypes = [P, I64, I64, I64, I, P, P]
            lib.oracle_epilogue_tokens.argtypes = [P, I64, I64, P, P, P, I, P]
            lib.oracle_fold_codes_asym.argtypes = [P, I64, I64, P, I, P, P, P]
            lib.oracle_rowsum.argtypes = [P, I64, I64, P]
            lib.oracle_epilogue_asym.argtypes = [P, P, P, I64, I64, P, P, I, P]
            lib.oracle_fold_layernorm.argtypes = [P, P, P, P, I64, P, P]
            lib.oracle_layernorm_quantize.argtypes = [P, I64, I64, I64, P, P, ctypes.c_float, I, P, P, P, P]
            lib.oracle_calibrate_clipped.argtypes = [P, I64, I64, I64, ctypes.c_double, P, P]
            lib.oracle_epilogue_quantize.argtypes = [P, I64, I64, P, P, I, P, P, I, P]
            for f in ("oracle_calibrate", "oracle_params", "oracle_fold", "oracle_quantize",
                      "oracle_matmul", "oracle_epilogue", "oracle_quantize_tokens", "oracle_epilogue_tokens",
                      "oracle_fold_codes_asym", "oracle_rowsum", "oracle_epilogue_asym",
                      "oracle_fold_layernorm", "oracle_layernorm_quantize", "oracle_calibrate_clipped",
                      "oracle_epilogue_quantize"):
                getattr(lib, f).restype = None
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != np.float16:
        raise TypeError(f"expected float16, got {a.dtype}")
    return a


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def qmax(bits: int) -> int:
    return (1 << (bits - 1)) - 1


def half_to_float(bits: np.ndarray) -> np.ndarray:
    """Binary16 bit patterns -> float32, element by element through the C oracle."""
    lib = _load()
    flat = np.ascontiguousarray(bits, dtype=np.uint16).ravel()
    return np.array([lib.ot_half_to_float(int(b)) for b in flat], dtype=np.float32).reshape(np.shape(bits))


def double_to_half(values: np.ndarray) -> np.ndarray:
    """float64 -> binary16 bit patterns (round half to even), through the C oracle."""
    lib = _load()
    flat = np.ascontiguousarray(values, dtype=np.float64).ravel()
    return np.array([lib.ot_double_to_half(float(v)) for v in flat], dtype=np.uint16).reshape(np.shape(values))


def calibrate(x: np.ndarray, mn: np.ndarray | None = None, mx: np.ndarray | None = None):
    """Per-channel (min, max) of fp16 X_cal[T, K]; pass mn/mx to continue a running calibration."""
    x = _f16(x)
    T, K = x.shape
    reset = mn is None
    mn = np.empty(K, np.float32) if reset else _f32(mn).copy()
    mx = np.empty(K, np.float32) if reset else _f32(mx).copy()
    _load().oracle_calibrate(_ptr(x), T, K, K, _ptr(mn), _ptr(mx), 1 if reset else 0)
    return mn, mx


def params(mn: np.ndarray, mx: np.ndarray, bits: int, symmetrize: bool = True):
    """(z, s, r) per channel: symmetrization factor, scale, reciprocal scale."""
    mn, mx = _f32(mn), _f32(mx)
    K = mn.shape[0]
    z, s, r = (np.empty(K, np.float32) for _ in range(3))
    _load().oracle_params(_ptr(mn), _ptr(mx), K, bits, 1 if symmetrize else 0, _ptr(z), _ptr(s), _ptr(r))
    return z, s, r


def fold(w: np.ndarray, b: np.ndarray | None, z: np.ndarray, s: np.ndarray, bits_w: int):
    """(qw int8 [N,K], sw fp32 [N], b' fp32 [N]) from fp16 W[N,K], fp16 b[N] (or None)."""
    w = _f16(w)
    N, K = w.shape
    z, s = _f32(z), _f32(s)
    bb = None if b is None else _f16(b)
    qw = np.empty((N, K), np.int8)
    sw = np.empty(N, np.float32)
    bf = np.empty(N, np.float32)
    _load().oracle_fold(_ptr(w), None if bb is None else _ptr(bb), N, K, _ptr(z), _ptr(s), bits_w,
                        _ptr(qw), _ptr(sw), _ptr(bf))
    return qw, sw, bf


def quantize(x: np.ndarray, z: np.ndarray, r: np.ndarray, bits_a: int) -> np.ndarray:
    """int8 codes [M, K] of fp16 X[M, K]."""
    x = _f16(x)
    M, K = x.shape
    q = np.empty((M, K), np.int8)
    _load().oracle_quantize(_ptr(x), M, K, K, _ptr(_f32(z)), _ptr(_f32(r)), bits_a, _ptr(q))
    return q


def matmul(q: np.ndarray, qw: np.ndarray) -> np.ndarray:
    """int64 acc[M, N] = q[M, K] . qw[N, K]^T."""
    q = np.ascontiguousarray(q, dtype=np.int8)
    qw = np.ascontiguousarray(qw, dtype=np.int8)
    M, K = q.shape
    N = qw.shape[0]
    assert qw.shape[1] == K
    acc = np.empty((M, N), np.int64)
    _load().oracle_matmul(_ptr(q), _ptr(qw), M, N, K, _ptr(acc))
    return acc


def epilogue(acc: np.ndarray, sw: np.ndarray, bfold: np.ndarray, relu: bool = False) -> np.ndarray:
    """fp16 Y[M, N] = fp16(fma((float)acc, sw, b')), optional ReLU."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    M, N = acc.shape
    y = np.empty((M, N), np.uint16)
    _load().oracle_epilogue(_ptr(acc), M, N, _ptr(_f32(sw)), _ptr(_f32(bfold)), 1 if relu else 0, _ptr(y))
    return y.view(np.float16)


def linear(x: np.ndarray, qw: np.ndarray, sw: np.ndarray, bfold: np.ndarray, z: np.ndarray,
           r: np.ndarray, bits_a: int, relu: bool = False):
    """Online path for one layer: codes, int64 accumulators and fp16 output."""
    q = quantize(x, z, r, bits_a)
    acc = matmul(q, qw)
    return q, acc, epilogue(acc, sw, bfold, relu)


def quantize_tokens(x: np.ndarray, bits_a: int):
    """(int8 codes [M, K], fp32 per-token scales [M]) of fp16 X (Eq. 3, Eq. 1 with z = 0)."""
    x = _f16(x)
    M, K = x.shape
    q = np.empty((M, K), np.int8)
    s = np.empty(M, np.float32)
    _load().oracle_quantize_tokens(_ptr(x), M, K, K, bits_a, _ptr(q), _ptr(s))
    return q, s


def quantize_weights(w: np.ndarray, bits_w: int):
    """(qw int8 [N, K], sw fp32 [N]): per-output-channel symmetric codes of W
    with no activation scale folded in (Eq. 3's W~): the fold with s = 1, z = 0."""
    w = _f16(w)
    K = w.shape[1]
    qw, sw, _ = fold(w, None, np.zeros(K, np.float32), np.ones(K, np.float32), bits_w)
    return qw, sw


def epilogue_tokens(acc: np.ndarray, s_tok: np.ndarray, sw: np.ndarray, bias: np.ndarray, relu: bool = False):
    """fp16 Y[M, N] = fp16(fma((float)acc, s_m * sw_n, b_n)), optional ReLU."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    M, N = acc.shape
    y = np.empty((M, N), np.uint16)
    _load().oracle_epilogue_tokens(_ptr(acc), M, N, _ptr(_f32(s_tok)), _ptr(_f32(sw)), _ptr(_f32(bias)),
                                   1 if relu else 0, _ptr(y))
    return y.view(np.float16)


def fold_codes_asym(w: np.ndarray, s: np.ndarray | None, bits_w: int):
    """Asymmetric per-output-channel codes of W_s = W (.) s (R9; s None: s = 1).
    Returns (qw int8 [N, K] stored as u - 2^(b-1), sw fp32 [N], zc int32 [N])."""
    w = _f16(w)
    N, K = w.shape
    ss = None if s is None else _f32(s)
    qw = np.empty((N, K), np.int8)
    sw = np.empty(N, np.float32)
    zc = np.empty(N, np.int32)
    _load().oracle_fold_codes_asym(_ptr(w), N, K, None if ss is None else _ptr(ss), bits_w, _ptr(qw), _ptr(sw),
                                   _ptr(zc))
    return qw, sw, zc


def rowsum(q: np.ndarray) -> np.ndarray:
    """int64 rs[m] = sum_k q[m, k]."""
    q = np.ascontiguousarray(q, dtype=np.int8)
    M, K = q.shape
    rs = np.empty(M, np.int64)
    _load().oracle_rowsum(_ptr(q), M, K, _ptr(rs))
    return rs


def epilogue_asym(acc: np.ndarray, rs: np.ndarray, zc: np.ndarray, sw: np.ndarray, bfold: np.ndarray,
                  relu: bool = False) -> np.ndarray:
    """fp16 Y[M, N] = fp16(fma((float)(acc - zc_n rs_m), sw_n, b'_n)), optional ReLU."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    rs = np.ascontiguousarray(rs, dtype=np.int64)
    zc = np.ascontiguousarray(zc, dtype=np.int32)
    M, N = acc.shape
    y = np.empty((M, N), np.uint16)
    _load().oracle_epilogue_asym(_ptr(acc), _ptr(rs), _ptr(zc), M, N, _ptr(_f32(sw)), _ptr(_f32(bfold)),
                                 1 if relu else 0, _ptr(y))
    return y.view(np.float16)


def fold_layernorm(gamma: np.ndarray, beta: np.ndarray, z: np.ndarray, r: np.ndarray):
    """(gamma_r, beta_r) fp32 [K]: gamma * r and (beta - z) * r (gamma, beta fp16)."""
    gamma, beta = _f16(gamma), _f16(beta)
    K = gamma.shape[0]
    gr, br = np.empty(K, np.float32), np.empty(K, np.float32)
    _load().oracle_fold_layernorm(_ptr(gamma), _ptr(beta), _ptr(_f32(z)), _ptr(_f32(r)), K, _ptr(gr), _ptr(br))
    return gr, br


def layernorm_quantize(h: np.ndarray, gamma_r: np.ndarray, beta_r: np.ndarray, eps: float, bits: int):
    """(codes int8 [M, K], rowsum int64 [M], mean fp32 [M], rstd fp32 [M]) of the
    LayerNorm of fp16 h [M, K] fused with the per-channel quantization."""
    h = _f16(h)
    M, K = h.shape
    q = np.empty((M, K), np.int8)
    rs = np.empty(M, np.int64)
    mean, rstd = np.empty(M, np.float32), np.empty(M, np.float32)
    _load().oracle_layernorm_quantize(_ptr(h), M, K, K, _ptr(_f32(gamma_r)), _ptr(_f32(beta_r)), float(eps), bits,
                                      _ptr(q), _ptr(rs), _ptr(mean), _ptr(rstd))
    return q, rs, mean, rstd


def calibrate_clipped(x: np.ndarray, alpha: float):
    """(lo, hi) fp32 [K]: per-channel order statistics of fp16 X_cal [T, K] at
    ascending ranks T' + 1 - ceil(alpha T') and ceil(alpha T') (NaN ignored)."""
    x = _f16(x)
    T, K = x.shape
    lo, hi = np.empty(K, np.float32), np.empty(K, np.float32)
    _load().oracle_calibrate_clipped(_ptr(x), T, K, K, float(alpha), _ptr(lo), _ptr(hi))
    return lo, hi


def epilogue_quantize(acc: np.ndarray, sw: np.ndarray, bfold: np.ndarray, z_next: np.ndarray, r_next: np.ndarray,
                      bits_next: int, relu: bool = False) -> np.ndarray:
    """int8 codes q'[M, N] = round((fma((float)acc, sw, b') [ReLU] - z') * r') of the next layer."""
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    M, N = acc.shape
    q = np.empty((M, N), np.int8)
    _load().oracle_epilogue_quantize(_ptr(acc), M, N, _ptr(_f32(sw)), _ptr(_f32(bfold)), 1 if relu else 0,
                                     _ptr(_f32(z_next)), _ptr(_f32(r_next)), bits_next, _ptr(q))
    return q


# ---------------------------------------------------------------------------
# Threaded drivers: the same C functions run on disjoint row (or channel)
# ranges in parallel threads (ctypes releases the GIL during each call).
# Every output element is computed by exactly the code above, so results are
# identical to the single-threaded calls; only the wall time changes.
# ---------------------------------------------------------------------------
def host_threads() -> int:
    """Cores this process may run on."""
    return len(os.sched_getaffinity(0))


def _ranges(n: int, parts: int):
    parts = max(1, min(parts, n))
    return [(n * i // parts, n * (i + 1) // parts) for i in range(parts)]


def _run_parallel(fn, ranges, threads):
    from concurrent.futures import ThreadPoolExecutor
    if len(ranges) <= 1:
        return [fn(*r) for r in ranges]
    with ThreadPoolExecutor(max_workers=threads) as ex:
        return list(ex.map(lambda r: fn(*r), ranges))


def calibrate_mt(x: np.ndarray, mn: np.ndarray | None = None, mx: np.ndarray | None = None,
                 threads: int | None = None):
    """calibrate() with the channels split over threads (each channel's min /
    max is one thread's sequential scan over the tokens, as in calibrate)."""
    x = _f16(x)
    T, K = x.shape
    threads = threads or host_threads()
    reset = mn is None
    mn = np.empty(K, np.float32) if reset else _f32(mn).copy()
    mx = np.empty(K, np.float32) if reset else _f32(mx).copy()
    lib = _load()
    base = x.ctypes.data

    def part(k0, k1):
        lib.oracle_calibrate(ctypes.c_void_p(base + 2 * k0), T, k1 - k0, K,
                             ctypes.c_void_p(mn.ctypes.data + 4 * k0), ctypes.c_void_p(mx.ctypes.data + 4 * k0),
                             1 if reset else 0)
    _run_parallel(part, _ranges(K, 4 * threads), threads)
    return mn, mx


def fold_mt(w: np.ndarray, b: np.ndarray | None, z: np.ndarray, s: np.ndarray, bits_w: int,
            threads: int | None = None):
    """fold() with the output channels (rows of W) split over threads; every
    row's codes, scale and folded bias depend on that row alone."""
    w = _f16(w)
    threads = threads or host_threads()
    parts = _run_parallel(lambda n0, n1: fold(w[n0:n1], None if b is None else b[n0:n1], z, s, bits_w),
                          _ranges(w.shape[0], 4 * threads), threads)
    return tuple(np.concatenate([p[i] for p in parts]) for i in range(3))


def quantize_mt(x: np.ndarray, z: np.ndarray, r: np.ndarray, bits_a: int, threads: int | None = None):
    """quantize() with the tokens split over threads."""
    x = _f16(x)
    threads = threads or host_threads()
    parts = _run_parallel(lambda m0, m1: quantize(x[m0:m1], z, r, bits_a), _ranges(x.shape[0], threads), threads)
    return np.concatenate(parts) if parts else np.empty((0, x.shape[1]), np.int8)


def matmul_mt(q: np.ndarray, qw: np.ndarray, threads: int | None = None) -> np.ndarray:
    """matmul() with the tokens (or, for few tokens, the output channels) split
    over threads; each accumulator is one thread's k-ascending int64 sum."""
    q = np.ascontiguousarray(q, dtype=np.int8)
    qw = np.ascontiguousarray(qw, dtype=np.int8)
    threads = threads or host_threads()
    M, N = q.shape[0], qw.shape[0]
    if M >= threads:
        parts = _run_parallel(lambda m0, m1: matmul(q[m0:m1], qw), _ranges(M, 4 * threads), threads)
        return np.concatenate(parts)
    parts = _run_parallel(lambda n0, n1: matmul(q, qw[n0:n1]), _ranges(N, 4 * threads), threads)
    return np.concatenate(parts, axis=1)


def epilogue_mt(acc: np.ndarray, sw: np.ndarray, bfold: np.ndarray, relu: bool = False,
                threads: int | None = None) -> np.ndarray:
    """epilogue() with the tokens split over threads."""
    threads = threads or host_threads()
    parts = _run_parallel(lambda m0, m1: epilogue(acc[m0:m1], sw, bfold, relu), _ranges(acc.shape[0], threads),
                          threads)
    return np.concatenate(parts)
