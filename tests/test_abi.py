"""The C-ABI library builds, loads and exports every function declared in
include/outliertune.h; host-side argument validation rejects bad requests
before anything is launched (no GPU needed for these calls)."""
import ctypes
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "outliertune.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(ot_\w+)\s*\(", text, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2406_18832_gb300 import build
    path = build.build()
    return ctypes.CDLL(path), path


def test_header_declares_the_boundary():
    names = declared_functions()
    for f in ("ot_calibrate", "ot_derive_params", "ot_fold_weights", "ot_quantize_act", "ot_linear",
              "ot_linear_s32", "ot_get_device_status", "ot_status_string", "ot_version"):
        assert f in names


def test_library_exports_every_declared_symbol(lib):
    handle, path = lib
    for name in declared_functions():
        assert hasattr(handle, name), name
    nm = shutil.which("nm")
    if nm:
        out = subprocess.run([nm, "-D", "--defined-only", path], capture_output=True, text=True).stdout
        exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
        for name in declared_functions():
            assert name in exported, name


def test_status_strings_and_version(lib):
    handle, _ = lib
    handle.ot_status_string.restype = ctypes.c_char_p
    handle.ot_status_string.argtypes = [ctypes.c_int]
    assert handle.ot_status_string(0) == b"OT_OK"
    assert b"TIMEOUT" in handle.ot_status_string(4)
    assert handle.ot_status_string(99) == b"unknown ot_status"
    assert handle.ot_version() >= 100


def _linear_args(handle):
    P, I64, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    S = ctypes.c_size_t
    handle.ot_linear.argtypes = [P, I, I64, I64, P, P, P, I64, I, I, P, I64, I, P, S, P]
    handle.ot_linear_s32.argtypes = [P, I, I64, I64, P, I64, I, I, P, P, S, P]
    handle.ot_quantize_act.argtypes = [P, I64, I64, I64, P, P, I, P, I, P]
    handle.ot_calibrate.argtypes = [P, I64, I64, I64, P, P, I, P]
    handle.ot_fold_weights.argtypes = [P, P, I, I, P, P, I64, I64, I, P, P, P, P, P, P, P]
    handle.ot_selftest_wait_timeout.argtypes = [I64, P]
    handle.ot_linear_asym.argtypes = [P, I64, I64, P, P, P, P, P, I64, I, I, P, I64, I, P, S, P]
    handle.ot_quantize_act_rowsum.argtypes = [P, I64, I64, I64, P, P, I, P, I, P, P]
    handle.ot_fold_weights_asym.argtypes = [P, P, I, I, P, P, I64, I64, I, P, P, P, P, P, P, P, P]
    handle.ot_linear_quantize_next.argtypes = [P, I64, I64, P, P, P, I64, I, I, I, P, P, I, P, I64, P, S, P]
    handle.ot_linear_fused.argtypes = [P, I64, I64, I64, P, P, I, P, P, P, I64, I, P, P, I64, I, I, P, S, P]


# Fake, 256-byte-aligned addresses: every call below must be rejected on the
# host before any CUDA call, so they are never dereferenced.
A = 0x10000000
A2 = A + 0x100000


def test_validation_rejects_bad_arguments_before_launch(lib):
    handle, _ = lib
    _linear_args(handle)
    INV, UNS = 1, 2
    # K not a multiple of 16
    assert handle.ot_linear(A, 1, 4, 24, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    # bits outside [2, 8]
    assert handle.ot_linear(A, 1, 4, 64, A2, A, A, 16, 9, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear(A, 1, 4, 64, A2, A, A, 16, 8, 1, A, 16, 0, None, 0, None) == INV
    # misaligned operands
    assert handle.ot_linear(A + 2, 1, 4, 64, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear(A, 1, 4, 64, A2 + 8, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    # null pointers, ldy < N, negative sizes
    assert handle.ot_linear(A, 1, 4, 64, None, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear(A, 1, 4, 64, A2, None, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear(A, 1, 4, 64, A2, A, A, 16, 8, 8, A, 8, 0, None, 0, None) == INV
    assert handle.ot_linear(A, 1, -1, 64, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    # K beyond the int32 accumulator for W8A8 (K * 127 * 127 >= 2^31)
    assert handle.ot_linear(A, 1, 4, 133152, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == UNS
    assert handle.ot_linear_s32(A, 1, 4, 24, A2, 16, 8, 8, A, None, 0, None) == INV
    # code format other than OT_CODE_I8 / OT_CODE_F16; int8 codes keep the same checks
    assert handle.ot_linear(A, 7, 4, 64, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear(A + 8, 0, 4, 64, A2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear_s32(A, 0, 4, 24, A2, 16, 8, 8, A, None, 0, None) == INV
    # workspace must be 16-byte aligned
    assert handle.ot_linear(A, 1, 4, 64, A2, A, A, 16, 8, 8, A, 16, 0, A + 8, 1 << 20, None) == INV
    # quantize: bad format, unaligned z, ldx < K
    assert handle.ot_quantize_act(A, 4, 64, 64, A, A, 8, A2, 7, None) == INV
    assert handle.ot_quantize_act(A, 4, 64, 64, A + 4, A, 8, A2, 1, None) == INV
    assert handle.ot_quantize_act(A, 4, 64, 32, A, A, 8, A2, 1, None) == INV
    # calibrate: K not a multiple of 8
    assert handle.ot_calibrate(A, 4, 12, 12, A, A, 1, None) == INV
    # fold: K not a multiple of 16, unaligned weights
    assert handle.ot_fold_weights(A, A, 8, 1, A, None, 16, 24, 8, A, A, A, A2, A, A, None) == INV
    assert handle.ot_fold_weights(A, A, 8, 1, A + 2, None, 16, 64, 8, A, A, A, A2, A, A, None) == INV
    # self-test limit outside [1 ms, 2 s]
    assert handle.ot_selftest_wait_timeout(10, None) == INV
    # asymmetric weights: null zero points / row sums, unaligned zero points
    assert handle.ot_linear_asym(A, 4, 64, A2, A, None, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear_asym(A, 4, 64, A2, A, A, None, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    assert handle.ot_linear_asym(A, 4, 64, A2, A, A + 2, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV
    # the corrected sum K * 127 * 255 must fit int32: K = 66,320 is refused, 66,304 is not
    assert handle.ot_linear_asym(A, 4, 66320, A2, A, A, A, A, 16, 8, 8, A, 16, 0, None, 0, None) == UNS
    assert 127 * 255 * 66304 < 2 ** 31
    assert handle.ot_quantize_act_rowsum(A, 4, 64, 64, A, A, 8, A2, 1, None, None) == INV
    assert handle.ot_quantize_act_rowsum(A, 4, 64, 64, A, A, 8, A2, 1, A + 2, None) == INV
    assert handle.ot_fold_weights_asym(A, A, 8, 1, A, None, 16, 64, 8, A, A, A, A2, A, None, A, None) == INV
    # chained epilogue: null / unaligned z', r', next bits outside [2, 8], ldq < N
    qn = handle.ot_linear_quantize_next
    assert qn(A, 4, 64, A2, A, A, 16, 8, 8, 1, None, A, 8, A, 16, None, 0, None) == INV
    assert qn(A, 4, 64, A2, A, A, 16, 8, 8, 1, A, A + 2, 8, A, 16, None, 0, None) == INV
    assert qn(A, 4, 64, A2, A, A, 16, 8, 8, 1, A, A, 9, A, 16, None, 0, None) == INV
    assert qn(A, 4, 64, A2, A, A, 16, 8, 8, 1, A, A, 8, A, 15, None, 0, None) == INV
    # fused quantize + linear: ldx < K, null z, unaligned x, null code buffer, unknown mode,
    # the in-producer form above 128 tokens
    fz = handle.ot_linear_fused
    assert fz(A, 4, 64, 56, A, A, 8, A2, A, A, 16, 8, A2, A, 16, 0, 0, None, 0, None) == INV
    assert fz(A, 4, 64, 64, None, A, 8, A2, A, A, 16, 8, A2, A, 16, 0, 0, None, 0, None) == INV
    assert fz(A + 8, 4, 64, 64, A, A, 8, A2, A, A, 16, 8, A2, A, 16, 0, 0, None, 0, None) == INV
    assert fz(A, 4, 64, 64, A, A, 8, A2, A, A, 16, 8, None, A, 16, 0, 0, None, 0, None) == INV
    assert fz(A, 4, 64, 64, A, A, 8, A2, A, A, 16, 8, A2, A, 16, 0, 3, None, 0, None) == INV
    assert fz(A, 129, 64, 64, A, A, 8, A2, A, A, 16, 8, A2, A, 16, 0, 1, None, 0, None) == UNS


def test_validation_of_the_layernorm_calibration_and_per_token_entry_points(lib):
    """Host-side checks of the remaining entry points, each rejected before any
    CUDA call: LayerNorm fusion, token-wise clipping, per-token quantization."""
    handle, _ = lib
    INV, UNS = 1, 2
    P, I64, I, S = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_size_t
    F, D = ctypes.c_float, ctypes.c_double
    handle.ot_layernorm_quantize.argtypes = [P, I64, I64, I64, P, P, F, I, P, I, P, P]
    handle.ot_fold_layernorm.argtypes = [P, P, P, P, I64, P, P, P]
    handle.ot_calibrate_clipped.argtypes = [P, I64, I64, I64, D, P, P, P]
    handle.ot_quantize_tokens.argtypes = [P, I64, I64, I64, I, P, I, P, P]
    handle.ot_quantize_weights.argtypes = [P, I64, I64, I, P, P, P]
    handle.ot_linear_per_token.argtypes = [P, I64, I64, P, P, P, P, I64, I, I, P, I64, I, P, S, P]
    handle.ot_derive_params.argtypes = [P, P, I64, I, I, P, P, P, P]
    nan = float("nan")
    ln = handle.ot_layernorm_quantize
    assert ln(A, 4, 12, 12, A, A, 1e-5, 8, A2, 1, None, None) == INV            # K % 8
    assert ln(A, 4, 64, 56, A, A, 1e-5, 8, A2, 1, None, None) == INV            # ldh < K
    assert ln(A, 4, 64, 64, A, A, 1e-5, 8, A2, 7, None, None) == INV            # code format
    assert ln(A, 4, 64, 64, A, A, nan, 8, A2, 1, None, None) == INV             # eps NaN
    assert ln(A, 4, 64, 64, A, A, -1.0, 8, A2, 1, None, None) == INV            # eps < 0
    assert ln(A, 4, 64, 64, None, A, 1e-5, 8, A2, 1, None, None) == INV         # gamma_r
    assert ln(A + 8, 4, 64, 64, A, A, 1e-5, 8, A2, 1, None, None) == INV        # h alignment
    assert ln(A, 4, 64, 64, A, A, 1e-5, 8, A2, 1, A + 2, None) == INV           # rowsum alignment
    assert ln(A, 4, 64, 64, A, A, 1e-5, 1, A2, 1, None, None) == INV            # bits
    big = (1 << 22) + 8
    assert ln(A, 4, big, big, A, A, 1e-5, 8, A2, 1, None, None) == UNS          # exact 64-bit sums bound
    fl = handle.ot_fold_layernorm
    assert fl(A, A, A, A, 0, A, A, None) == INV
    assert fl(None, A, A, A, 64, A, A, None) == INV
    assert fl(A, A, A, A, 64, A + 2, A, None) == INV
    assert fl(A, A, A, A, 1 << 31, A, A, None) == UNS
    cc = handle.ot_calibrate_clipped
    assert cc(A, 16, 64, 64, 0.0, A, A, None) == INV
    assert cc(A, 16, 64, 64, 1.5, A, A, None) == INV
    assert cc(A, 16, 64, 64, nan, A, A, None) == INV
    assert cc(A, 16, 64, 64, 0.99, None, A, None) == INV
    assert cc(A, 16, 64, 32, 0.99, A, A, None) == INV
    assert cc(A, 1 << 31, 64, 64, 0.99, A, A, None) == UNS
    qt = handle.ot_quantize_tokens
    assert qt(A, 4, 64, 64, 8, A2, 7, A, None) == INV
    assert qt(A, 4, 64, 64, 8, A2, 1, None, None) == INV
    assert qt(A, 4, 12, 12, 8, A2, 1, A, None) == INV
    assert qt(A, 1 << 31, 64, 64, 8, A2, 1, A, None) == UNS
    qwf = handle.ot_quantize_weights
    assert qwf(A, 16, 24, 8, A2, A, None) == INV
    assert qwf(A, 16, 64, 8, A2, None, None) == INV
    pt = handle.ot_linear_per_token
    assert pt(A, 4, 64, A2, A, None, A, 16, 8, 8, A, 16, 0, None, 0, None) == INV  # s_tok
    assert pt(A, 4, 64, A2, A, A, None, 16, 8, 8, A, 16, 0, None, 0, None) == INV  # bias
    assert pt(A, 4, 64, A2, A, A, A, 16, 8, 8, A, 8, 0, None, 0, None) == INV     # ldy < N
    dp = handle.ot_derive_params
    assert dp(A, A, 0, 8, 1, A, A, A, None) == INV
    assert dp(A, A, 64, 8, 1, A, None, A, None) == INV
    assert dp(A, A, 64, 1, 1, A, A, A, None) == INV


def test_binding_refuses_host_tensors():
    import torch
    from paper_2406_18832_gb300 import binding
    q = torch.zeros(4, 64, dtype=torch.float16)
    qw = torch.zeros(16, 64, dtype=torch.int8)
    with pytest.raises((ValueError, RuntimeError)):
        binding.ot_linear(q, qw, torch.ones(16), torch.zeros(16), 8, 8, torch.empty(4, 16, dtype=torch.float16))
