// api.cu -- the C ABI (include/outliertune.h): argument validation on the
// host, then one or two kernel launches on the caller's stream.  Nothing here
// allocates device memory.
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "outliertune.h"
#include "ot_kernels.h"

namespace ot {

int num_sms() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
    if (dev < 64 && cache[dev]) return cache[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    if (dev < 64) cache[dev] = n;
    return n;
}

}  // namespace ot

namespace {

constexpr int kVersion = 100;  // 0.1.0

inline bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
inline bool bits_ok(int b) { return b >= 2 && b <= 8; }
inline int64_t qmax_of(int b) { return (int64_t(1) << (b - 1)) - 1; }
inline ot_status from_cuda(cudaError_t e) { return e == cudaSuccess ? OT_OK : OT_ERR_CUDA; }
inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }
constexpr int64_t kIntMax = 2147483647;

}  // namespace

extern "C" {

const char *ot_status_string(ot_status st) {
    switch (st) {
        case OT_OK: return "OT_OK";
        case OT_ERR_INVALID_ARG: return "OT_ERR_INVALID_ARG: invalid argument (pointer, size, alignment or bits)";
        case OT_ERR_UNSUPPORTED: return "OT_ERR_UNSUPPORTED: request outside what this build runs";
        case OT_ERR_CUDA: return "OT_ERR_CUDA: a CUDA call or kernel launch failed";
        case OT_ERR_TIMEOUT: return "OT_ERR_TIMEOUT: a bounded device wait gave up";
        case OT_ERR_BOUNDS: return "OT_ERR_BOUNDS: a kernel index check failed (debug build)";
    }
    return "unknown ot_status";
}

int ot_version(void) { return kVersion; }

int ot_debug_build(void) {
#ifdef OT_DEBUG
    return 1;
#else
    return 0;
#endif
}

ot_status ot_calibrate(const void *x_f16, int64_t T, int64_t K, int64_t ldx, float *ch_min, float *ch_max,
                       int reset, void *stream) {
    if (T < 0 || K <= 0 || K % 8 != 0 || ldx < K || ldx % 8 != 0) return OT_ERR_INVALID_ARG;
    if (!ch_min || !ch_max || !aligned(ch_min, 4) || !aligned(ch_max, 4)) return OT_ERR_INVALID_ARG;
    if (T > 0 && (!x_f16 || !aligned(x_f16, 16))) return OT_ERR_INVALID_ARG;
    if (T > kIntMax * 64) return OT_ERR_UNSUPPORTED;
    return from_cuda(ot::launch_calibrate(x_f16, T, K, ldx, ch_min, ch_max, reset, as_stream(stream)));
}

ot_status ot_calibrate_clipped(const void *x_f16, int64_t T, int64_t K, int64_t ldx, double alpha, float *ch_lo,
                               float *ch_hi, void *stream) {
    if (T < 0 || K <= 0 || ldx < K || !(alpha > 0.0) || !(alpha <= 1.0)) return OT_ERR_INVALID_ARG;
    if (!ch_lo || !ch_hi || !aligned(ch_lo, 4) || !aligned(ch_hi, 4)) return OT_ERR_INVALID_ARG;
    if (T > 0 && (!x_f16 || !aligned(x_f16, 2))) return OT_ERR_INVALID_ARG;
    if (T > kIntMax) return OT_ERR_UNSUPPORTED;  // 32-bit histogram counts
    return from_cuda(ot::launch_calibrate_clipped(x_f16, T, K, ldx, alpha, ch_lo, ch_hi, as_stream(stream)));
}

ot_status ot_derive_params(const float *ch_min, const float *ch_max, int64_t K, int bits_a, int symmetrize,
                           float *z, float *s, float *r, void *stream) {
    if (K <= 0 || !bits_ok(bits_a)) return OT_ERR_INVALID_ARG;
    if (!ch_min || !ch_max || !z || !s || !r) return OT_ERR_INVALID_ARG;
    return from_cuda(ot::launch_params(ch_min, ch_max, K, bits_a, symmetrize, z, s, r, as_stream(stream)));
}

ot_status ot_fold_weights(const float *ch_min, const float *ch_max, int bits_a, int symmetrize, const void *w_f16,
                          const void *b_f16, int64_t N, int64_t K, int bits_w, float *z, float *s, float *r,
                          int8_t *qw, float *sw, float *b_fold, void *stream) {
    if (N < 0 || K <= 0 || K % 16 != 0 || !bits_ok(bits_a) || !bits_ok(bits_w)) return OT_ERR_INVALID_ARG;
    if (!ch_min || !ch_max || !z || !s || !r || !sw || !b_fold) return OT_ERR_INVALID_ARG;
    if (N > 0 && (!w_f16 || !qw || !aligned(w_f16, 16) || !aligned(qw, 16))) return OT_ERR_INVALID_ARG;
    if (b_f16 && !aligned(b_f16, 2)) return OT_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    cudaError_t e = ot::launch_params(ch_min, ch_max, K, bits_a, symmetrize, z, s, r, st);
    if (e != cudaSuccess) return OT_ERR_CUDA;
    return from_cuda(ot::launch_fold(w_f16, b_f16, N, K, z, s, bits_w, qw, sw, b_fold, st));
}

ot_status ot_fold_weights_asym(const float *ch_min, const float *ch_max, int bits_a, int symmetrize,
                               const void *w_f16, const void *b_f16, int64_t N, int64_t K, int bits_w, float *z,
                               float *s, float *r, int8_t *qw, float *sw, int32_t *zc, float *b_fold, void *stream) {
    if (N < 0 || K <= 0 || K % 16 != 0 || !bits_ok(bits_a) || !bits_ok(bits_w)) return OT_ERR_INVALID_ARG;
    if (!ch_min || !ch_max || !z || !s || !r || !sw || !b_fold) return OT_ERR_INVALID_ARG;
    if (N > 0 && (!w_f16 || !qw || !zc || !aligned(w_f16, 16) || !aligned(qw, 16) || !aligned(zc, 4)))
        return OT_ERR_INVALID_ARG;
    if (b_f16 && !aligned(b_f16, 2)) return OT_ERR_INVALID_ARG;
    cudaStream_t st = as_stream(stream);
    cudaError_t e = ot::launch_params(ch_min, ch_max, K, bits_a, symmetrize, z, s, r, st);
    if (e != cudaSuccess) return OT_ERR_CUDA;
    return from_cuda(ot::launch_fold_asym(w_f16, b_f16, N, K, z, s, bits_w, qw, sw, zc, b_fold, st));
}

ot_status ot_quantize_act_rowsum(const void *x_f16, int64_t M, int64_t K, int64_t ldx, const float *z,
                                 const float *r, int bits_a, void *q, int q_format, int32_t *rowsum,
                                 void *stream) {
    if (M < 0 || K <= 0 || K % 8 != 0 || ldx < K || ldx % 8 != 0 || !bits_ok(bits_a)) return OT_ERR_INVALID_ARG;
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    if (!z || !r || !aligned(z, 16) || !aligned(r, 16)) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!x_f16 || !q || !rowsum || !aligned(x_f16, 16) || !aligned(q, 16) || !aligned(rowsum, 4)))
        return OT_ERR_INVALID_ARG;
    if ((M + 63) / 64 > 65535) return OT_ERR_UNSUPPORTED;
    if (K * qmax_of(bits_a) > kIntMax) return OT_ERR_UNSUPPORTED;  // int32 row sums
    return from_cuda(
        ot::launch_quantize(x_f16, M, K, ldx, z, r, bits_a, q, q_format, as_stream(stream), rowsum));
}

ot_status ot_fold_layernorm(const void *gamma_f16, const void *beta_f16, const float *z, const float *r, int64_t K,
                            float *gamma_r, float *beta_r, void *stream) {
    if (K <= 0 || !gamma_f16 || !beta_f16 || !z || !r || !gamma_r || !beta_r) return OT_ERR_INVALID_ARG;
    if (!aligned(gamma_f16, 2) || !aligned(beta_f16, 2) || !aligned(z, 4) || !aligned(r, 4) ||
        !aligned(gamma_r, 4) || !aligned(beta_r, 4))
        return OT_ERR_INVALID_ARG;
    if (K > kIntMax) return OT_ERR_UNSUPPORTED;
    return from_cuda(ot::launch_fold_layernorm(gamma_f16, beta_f16, z, r, K, gamma_r, beta_r, as_stream(stream)));
}

ot_status ot_layernorm_quantize(const void *h_f16, int64_t M, int64_t K, int64_t ldh, const float *gamma_r,
                                const float *beta_r, float eps, int bits_a, void *q, int q_format,
                                int32_t *rowsum, void *stream) {
    if (M < 0 || K <= 0 || K % 8 != 0 || ldh < K || ldh % 8 != 0 || !bits_ok(bits_a)) return OT_ERR_INVALID_ARG;
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    if (!(eps >= 0.0f) || !(eps < 3.0e38f)) return OT_ERR_INVALID_ARG;  // finite, non-negative (rejects NaN)
    if (!gamma_r || !beta_r || !aligned(gamma_r, 16) || !aligned(beta_r, 16)) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!h_f16 || !q || !aligned(h_f16, 16) || !aligned(q, 16))) return OT_ERR_INVALID_ARG;
    if (rowsum && !aligned(rowsum, 4)) return OT_ERR_INVALID_ARG;
    if (K > ((int64_t)1 << 22)) return OT_ERR_UNSUPPORTED;  // exact 64-bit partial sums of the squares
    return from_cuda(ot::launch_layernorm_quantize(h_f16, M, K, ldh, gamma_r, beta_r, eps, bits_a, q, q_format,
                                                   rowsum, as_stream(stream)));
}

ot_status ot_quantize_act(const void *x_f16, int64_t M, int64_t K, int64_t ldx, const float *z, const float *r,
                          int bits_a, void *q, int q_format, void *stream) {
    if (M < 0 || K <= 0 || K % 8 != 0 || ldx < K || ldx % 8 != 0 || !bits_ok(bits_a)) return OT_ERR_INVALID_ARG;
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    if (!z || !r || !aligned(z, 16) || !aligned(r, 16)) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!x_f16 || !q || !aligned(x_f16, 16) || !aligned(q, 16))) return OT_ERR_INVALID_ARG;
    if ((M + 63) / 64 > 65535) return OT_ERR_UNSUPPORTED;
    return from_cuda(ot::launch_quantize(x_f16, M, K, ldx, z, r, bits_a, q, q_format, as_stream(stream)));
}

ot_status ot_quantize_tokens(const void *x_f16, int64_t M, int64_t K, int64_t ldx, int bits_a, void *q,
                             int q_format, float *s_tok, void *stream) {
    if (M < 0 || K <= 0 || K % 8 != 0 || ldx < K || ldx % 8 != 0 || !bits_ok(bits_a)) return OT_ERR_INVALID_ARG;
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!x_f16 || !q || !s_tok || !aligned(x_f16, 16) || !aligned(q, 16) || !aligned(s_tok, 4)))
        return OT_ERR_INVALID_ARG;
    if (M > kIntMax) return OT_ERR_UNSUPPORTED;
    return from_cuda(ot::launch_quantize_tokens(x_f16, M, K, ldx, bits_a, q, q_format, s_tok, as_stream(stream)));
}

ot_status ot_quantize_weights(const void *w_f16, int64_t N, int64_t K, int bits_w, int8_t *qw, float *sw,
                              void *stream) {
    if (N < 0 || K <= 0 || K % 16 != 0 || !bits_ok(bits_w)) return OT_ERR_INVALID_ARG;
    if (N > 0 && (!w_f16 || !qw || !sw || !aligned(w_f16, 16) || !aligned(qw, 16))) return OT_ERR_INVALID_ARG;
    return from_cuda(ot::launch_quantize_weights(w_f16, N, K, bits_w, qw, sw, as_stream(stream)));
}

static ot_status linear_common(const void *q_f16, int64_t M, int64_t K, const int8_t *qw, int64_t N, int bits_a,
                               int bits_w, const void *out) {
    if (M < 0 || N <= 0 || K <= 0 || K % 16 != 0 || !bits_ok(bits_a) || !bits_ok(bits_w))
        return OT_ERR_INVALID_ARG;
    if (!qw || !aligned(qw, 16)) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!q_f16 || !aligned(q_f16, 16) || !out)) return OT_ERR_INVALID_ARG;
    if (M > kIntMax || N > kIntMax || K > kIntMax) return OT_ERR_UNSUPPORTED;
    if (K * qmax_of(bits_a) * qmax_of(bits_w) > kIntMax) return OT_ERR_UNSUPPORTED;  // int32 accumulator
    return OT_OK;
}

ot_status ot_linear_workspace_size(size_t *bytes) {
    if (!bytes) return OT_ERR_INVALID_ARG;
    *bytes = ot::linear_workspace_bytes();
    return OT_OK;
}

ot_status ot_linear(const void *q, int q_format, int64_t M, int64_t K, const int8_t *qw, const float *sw,
                    const float *b_fold, int64_t N, int bits_a, int bits_w, void *y_f16, int64_t ldy, int relu,
                    void *workspace, size_t workspace_bytes, void *stream) {
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    ot_status v = linear_common(q, M, K, qw, N, bits_a, bits_w, y_f16);
    if (v != OT_OK) return v;
    if (!sw || !b_fold || ldy < N || (y_f16 && !aligned(y_f16, 2))) return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    if (ldy > kIntMax) return OT_ERR_UNSUPPORTED;
    ot::LinearArgs a{q, qw, sw, b_fold, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                     workspace, workspace ? workspace_bytes : 0};
    a.q_fmt = q_format == OT_CODE_I8 ? ot::kCodesI8 : ot::kCodesF16;
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_linear_per_token(const void *q_f16, int64_t M, int64_t K, const int8_t *qw, const float *sw,
                              const float *s_tok, const float *bias, int64_t N, int bits_a, int bits_w, void *y_f16,
                              int64_t ldy, int relu, void *workspace, size_t workspace_bytes, void *stream) {
    ot_status v = linear_common(q_f16, M, K, qw, N, bits_a, bits_w, y_f16);
    if (v != OT_OK) return v;
    if (!sw || !bias || ldy < N || (y_f16 && !aligned(y_f16, 2))) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!s_tok || !aligned(s_tok, 4))) return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    if (ldy > kIntMax) return OT_ERR_UNSUPPORTED;
    ot::LinearArgs a{q_f16, qw, sw, bias, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                     workspace, workspace ? workspace_bytes : 0, s_tok};
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_linear_asym(const void *q_f16, int64_t M, int64_t K, const int8_t *qw, const float *sw,
                         const int32_t *zc, const int32_t *rowsum, const float *b_fold, int64_t N, int bits_a,
                         int bits_w, void *y_f16, int64_t ldy, int relu, void *workspace, size_t workspace_bytes,
                         void *stream) {
    ot_status v = linear_common(q_f16, M, K, qw, N, bits_a, bits_w, y_f16);
    if (v != OT_OK) return v;
    if (!sw || !b_fold || !zc || !aligned(zc, 4) || ldy < N || (y_f16 && !aligned(y_f16, 2)))
        return OT_ERR_INVALID_ARG;
    if (M > 0 && (!rowsum || !aligned(rowsum, 4))) return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    if (ldy > kIntMax) return OT_ERR_UNSUPPORTED;
    // the corrected sum, sum_k q (qw - zc) with |qw - zc| <= 2^bits_w - 1, must fit int32
    // (it bounds the stored codes' sum too: |qw| <= 2^(bits_w - 1))
    if (K * qmax_of(bits_a) * (2 * qmax_of(bits_w) + 1) > kIntMax) return OT_ERR_UNSUPPORTED;
    ot::LinearArgs a{q_f16, qw, sw, b_fold, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                     workspace, workspace ? workspace_bytes : 0, nullptr, zc, rowsum};
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_linear_fused(const void *x_f16, int64_t M, int64_t K, int64_t ldx, const float *z, const float *r,
                          int bits_a, const int8_t *qw, const float *sw, const float *b_fold, int64_t N, int bits_w,
                          void *q_f16, void *y_f16, int64_t ldy, int relu, int mode, void *workspace,
                          size_t workspace_bytes, void *stream) {
    if (mode != OT_FUSE_AUTO && mode != OT_FUSE_PRODUCER && mode != OT_FUSE_PDL) return OT_ERR_INVALID_ARG;
    if (ldx < K || ldx % 8 != 0) return OT_ERR_INVALID_ARG;
    ot_status v = linear_common(q_f16, M, K, qw, N, bits_a, bits_w, y_f16);
    if (v != OT_OK) return v;
    if (!z || !r || !aligned(z, 16) || !aligned(r, 16)) return OT_ERR_INVALID_ARG;
    if (M > 0 && (!x_f16 || !aligned(x_f16, 16))) return OT_ERR_INVALID_ARG;
    if (!sw || !b_fold || ldy < N || (y_f16 && !aligned(y_f16, 2))) return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    if (ldy > kIntMax || (M + 63) / 64 > 65535) return OT_ERR_UNSUPPORTED;
    if (M == 0) return OT_OK;
    const cudaStream_t st = as_stream(stream);
    if (mode == OT_FUSE_PRODUCER && M > ot::kFusedInKernelMaxTokens) return OT_ERR_UNSUPPORTED;
    if (mode == OT_FUSE_PRODUCER) {
        // the linear's token producer quantizes X itself (no codes in HBM)
        ot::LinearArgs a{x_f16, qw, sw, b_fold, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                         workspace, workspace ? workspace_bytes : 0};
        a.q_fmt = ot::kActF16;
        a.xz = z;
        a.xr = r;
        a.ldx = ldx;
        a.qmax_in = (int)qmax_of(bits_a);
        return from_cuda(ot::launch_linear(a, st));
    }
    cudaError_t e = ot::launch_quantize(x_f16, M, K, ldx, z, r, bits_a, q_f16, OT_CODE_F16, st);
    if (e != cudaSuccess) return from_cuda(e);
    ot::LinearArgs a{q_f16, qw, sw, b_fold, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                     workspace, workspace ? workspace_bytes : 0};
    a.weights_early = true;  // the quantize kernel releases the linear only after every earlier kernel ended
    return from_cuda(ot::launch_linear(a, st));
}

ot_status ot_linear_quantize_next(const void *q_f16, int64_t M, int64_t K, const int8_t *qw, const float *sw,
                                  const float *b_fold, int64_t N, int bits_a, int bits_w, int relu,
                                  const float *z_next, const float *r_next, int bits_next, void *q_next_f16,
                                  int64_t ldq, void *workspace, size_t workspace_bytes, void *stream) {
    ot_status v = linear_common(q_f16, M, K, qw, N, bits_a, bits_w, q_next_f16);
    if (v != OT_OK) return v;
    if (!sw || !b_fold || !z_next || !r_next || !bits_ok(bits_next) || ldq < N) return OT_ERR_INVALID_ARG;
    if (!aligned(z_next, 4) || !aligned(r_next, 4) || (q_next_f16 && !aligned(q_next_f16, 2)))
        return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    if (ldq > kIntMax) return OT_ERR_UNSUPPORTED;
    ot::LinearArgs a{q_f16, qw, sw, b_fold, q_next_f16, M, N, K, ldq, bits_a, bits_w, relu ? 1 : 0, false,
                     workspace, workspace ? workspace_bytes : 0, nullptr, nullptr, nullptr, z_next, r_next,
                     (int)qmax_of(bits_next)};
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_linear_noalloc(const void *q_f16, int64_t M, int64_t K, const int8_t *qw, const float *sw,
                            const float *b_fold, int64_t N, int bits_a, int bits_w, void *y_f16, int64_t ldy,
                            int relu, void *stream) {
    ot_status v = linear_common(q_f16, M, K, qw, N, bits_a, bits_w, y_f16);
    if (v != OT_OK) return v;
    if (!sw || !b_fold || ldy < N || (y_f16 && !aligned(y_f16, 2))) return OT_ERR_INVALID_ARG;
    if (ldy > kIntMax) return OT_ERR_UNSUPPORTED;
    // the device's stream-K layout must fit the fixed scratch array
    if (ot::linear_workspace_bytes() > ot::kNoAllocScratchBytes) return OT_ERR_UNSUPPORTED;
    void *scratch = nullptr;
    if (ot::noalloc_scratch(&scratch, as_stream(stream)) != cudaSuccess) return OT_ERR_CUDA;
    ot::LinearArgs a{q_f16, qw, sw, b_fold, y_f16, M, N, K, ldy, bits_a, bits_w, relu ? 1 : 0, false,
                     scratch, ot::kNoAllocScratchBytes};
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_linear_s32(const void *q, int q_format, int64_t M, int64_t K, const int8_t *qw, int64_t N,
                        int bits_a, int bits_w, int32_t *acc, void *workspace, size_t workspace_bytes,
                        void *stream) {
    if (q_format != OT_CODE_I8 && q_format != OT_CODE_F16) return OT_ERR_INVALID_ARG;
    ot_status v = linear_common(q, M, K, qw, N, bits_a, bits_w, acc);
    if (v != OT_OK) return v;
    if (acc && !aligned(acc, 4)) return OT_ERR_INVALID_ARG;
    if (workspace && !aligned(workspace, 16)) return OT_ERR_INVALID_ARG;
    ot::LinearArgs a{q, qw, nullptr, nullptr, acc, M, N, K, N, bits_a, bits_w, 0, true,
                     workspace, workspace ? workspace_bytes : 0};
    a.q_fmt = q_format == OT_CODE_I8 ? ot::kCodesI8 : ot::kCodesF16;
    return from_cuda(ot::launch_linear(a, as_stream(stream)));
}

ot_status ot_selftest_wait_timeout(int64_t limit_ns, void *stream) {
    if (limit_ns < 1000000 || limit_ns > 2000000000) return OT_ERR_INVALID_ARG;
    return from_cuda(ot::launch_wait_timeout(limit_ns, as_stream(stream)));
}

ot_status ot_get_device_status(void *stream) {
    int v = 0;
    if (ot::read_clear_status(&v, as_stream(stream)) != cudaSuccess) return OT_ERR_CUDA;
#ifdef OT_DEBUG
    // the first failed index check of each file's kernels (source line, 0 = none)
    unsigned lines[4] = {0, 0, 0, 0};
    if (ot::dbg_read_clear_gemm(&lines[0]) != cudaSuccess || ot::dbg_read_clear_gemv(&lines[1]) != cudaSuccess ||
        ot::dbg_read_clear_quant(&lines[2]) != cudaSuccess || ot::dbg_read_clear_fold(&lines[3]) != cudaSuccess)
        return OT_ERR_CUDA;
    for (unsigned l : lines)
        if (l != 0) return OT_ERR_BOUNDS;
#endif
    return v == OT_ERR_TIMEOUT ? OT_ERR_TIMEOUT : OT_OK;
}

}  // extern "C"
