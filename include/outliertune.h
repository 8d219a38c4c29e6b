/*
 * outliertune.h -- C ABI of the GB300 (sm_103a) per-channel quantized linear
 * layer of OutlierTune (arXiv 2406.18832).
 *
 * The method: activations X are symmetrized per input channel (X_hat = X - z,
 * Section 3.2) and quantized per channel with static scales s (Eq. 6); the
 * weights absorb the activation scales before they are quantized per output
 * channel ("pre-execution of dequantization", Eq. 5, Eq. 6); the integer
 * product is rescaled per output channel only and the symmetrization shift
 * comes back through the bias b' = b + z W^T (Eq. 7).
 *
 * Conventions shared by every entry point
 *   - Every pointer is DEVICE memory owned by the caller, unless stated.  The
 *     library allocates no device memory and keeps no per-call state.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued asynchronously; outputs are valid once the
 *     stream has reached that point.  Nothing here synchronizes the stream
 *     except ot_get_device_status and the first ot_linear_noalloc call on a
 *     device.
 *   - Layouts are row-major.  X is [tokens, K] with row stride ldx elements,
 *     W is [N, K] (out x in, the nn.Linear layout that Eq. 6's W^T implies),
 *     Y is [M, N] with row stride ldy elements.
 *   - bits (bits_a for activations, bits_w for weights) is in [2, 8];
 *     qmax = 2^(bits-1) - 1 and codes lie in [-qmax, qmax] (127 for Int8,
 *     31 for Int6).  Rounding is round-half-to-even in fp32.
 *   - Argument errors are detected on the host before anything is launched
 *     and return OT_ERR_INVALID_ARG or OT_ERR_UNSUPPORTED; a failed launch
 *     returns OT_ERR_CUDA.  No exception crosses the ABI.  Device-side waits
 *     are bounded: a wait that gives up records OT_ERR_TIMEOUT in a device
 *     status word that ot_get_device_status reads.
 */
#ifndef OUTLIERTUNE_H
#define OUTLIERTUNE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    OT_OK = 0,
    OT_ERR_INVALID_ARG = 1,  /* null pointer, bad size, alignment or bits */
    OT_ERR_UNSUPPORTED = 2,  /* valid request this build does not run (e.g. K too large) */
    OT_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed */
    OT_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up */
    OT_ERR_BOUNDS = 5        /* debug builds only (OT_DEBUG): a kernel's index
                                check failed and the access was skipped */
} ot_status;

/* Storage format of activation codes (written by the quantize entry points,
 * read by ot_linear / ot_linear_s32). */
typedef enum {
    OT_CODE_I8 = 0,   /* int8 codes, 1 byte per element (the paper's storage) */
    OT_CODE_F16 = 1   /* the same integers stored exactly as fp16: the operand
                         format of the tensor cores (sm_103a has no integer
                         tcgen05 MMA, so the product runs on the fp16 tensor
                         path); the fastest input for more than 128 tokens */
} ot_code_format;

/* Human-readable name of a status code (static string, never NULL). */
const char *ot_status_string(ot_status st);

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
int ot_version(void);

/* 1 when the library was compiled with OT_DEBUG (kernels check their global
 * indices against the sizes they were given, skip an access that fails and
 * report it through ot_get_device_status as OT_ERR_BOUNDS), else 0.  The paper
 * has no counterpart: it stands in for a memory checker. */
int ot_debug_build(void);

/*
 * ot_calibrate -- per-channel running min / max of calibration activations
 * (Appendix A "min-max calibration"; the max and min of Section 3.2).
 *   x_f16   fp16 [T, K], row stride ldx elements (ldx >= K); 16-byte aligned,
 *           K and ldx multiples of 8.
 *   ch_min, ch_max  fp32 [K], in/out.  reset != 0 first sets them to
 *           (+inf, -inf); reset == 0 folds this batch into their current
 *           values, so a calibration set can be streamed batch by batch.
 *   NaN inputs are ignored.  T == 0 only applies the reset.
 */
ot_status ot_calibrate(const void *x_f16, int64_t T, int64_t K, int64_t ldx,
                       float *ch_min, float *ch_max, int reset, void *stream);

/*
 * ot_derive_params -- symmetrization factor and static scale per channel
 * (Section 3.2; Eq. 1 with zero point 0):
 *   z = (max + min) / 2, amp = max(max - z, z - min),
 *   s = amp / qmax, r = qmax / amp            (fp32, IEEE division)
 * symmetrize == 0 gives the Table 6 "Non-Sym" variant: z = 0,
 * amp = max(|max|, |min|).  A channel with amp == 0, or without finite
 * calibration data, gets s = r = 0 (its codes are 0; a constant channel is
 * then carried exactly by z through the folded bias).
 *   ch_min, ch_max  fp32 [K] in;  z, s, r  fp32 [K] out.
 */
ot_status ot_derive_params(const float *ch_min, const float *ch_max, int64_t K,
                           int bits_a, int symmetrize, float *z, float *s,
                           float *r, void *stream);

/*
 * ot_fold_weights -- pre-execution of dequantization and bias correction,
 * done once per layer (Eq. 5, Eq. 6 right-hand side, Eq. 7; Section 3.2
 * "predetermined offline"):
 *   W_s[n,k] = W[n,k] * s_k                              (fp32)
 *   sw_n = max_k |W_s[n,k]| / qmax_w,  rw_n = qmax_w / max_k |W_s[n,k]|
 *   qw[n,k] = round(W_s[n,k] * rw_n)  in [-qmax_w, qmax_w]
 *   b'_n = b_n + sum_k z_k W[n,k]       (fp64, k ascending, rounded to fp32)
 * The parameters z, s, r come from (ch_min, ch_max) as in ot_derive_params
 * and are written out as well.
 *   ch_min, ch_max fp32 [K] in; w_f16 fp16 [N, K] (16-byte aligned, K % 16 == 0);
 *   b_f16 fp16 [N] or NULL (no bias);  z, s, r fp32 [K] out;
 *   qw int8 [N, K] out (16-byte aligned);  sw fp32 [N] out;  b_fold fp32 [N] out.
 */
ot_status ot_fold_weights(const float *ch_min, const float *ch_max, int bits_a,
                          int symmetrize, const void *w_f16, const void *b_f16,
                          int64_t N, int64_t K, int bits_w, float *z, float *s,
                          float *r, int8_t *qw, float *sw, float *b_fold,
                          void *stream);

/*
 * ot_quantize_act -- symmetrize and quantize activations per channel with
 * the static parameters (round(X_hat / s) of Eq. 6 / Eq. 7):
 *   q[m,k] = clamp(round_half_even((x[m,k] - z_k) * r_k), -qmax_a, qmax_a)
 * evaluated in fp32 (subtract, multiply, round: two roundings as written).
 * NaN gives code 0, +-inf and out-of-range values saturate.
 *   x_f16   fp16 [M, K], row stride ldx (16-byte aligned; K, ldx % 8 == 0)
 *   z, r    fp32 [K]
 *   q       [M, K] dense, int8 (OT_CODE_I8) or fp16 (OT_CODE_F16); 16-byte aligned
 */
ot_status ot_quantize_act(const void *x_f16, int64_t M, int64_t K, int64_t ldx,
                          const float *z, const float *r, int bits_a, void *q,
                          int q_format, void *stream);

/*
 * ot_linear -- the quantized linear with external per-output-channel scaling
 * (Eq. 6) and the folded bias (Eq. 7):
 *   acc[m,n] = sum_k q[m,k] * qw[n,k]            exact integer
 *   y[m,n]   = fp16( fma((float)acc[m,n], sw_n, b'_n) ), then ReLU if relu != 0
 *   q       activation codes [M, K], dense, |q| <= qmax(bits_a); 16-byte
 *           aligned, K % 16 == 0; q_format OT_CODE_I8 (int8, as ot_quantize_act
 *           writes them with OT_CODE_I8) or OT_CODE_F16 (fp16 integers).  int8
 *           codes are widened to fp16 inside the kernel (decode kernel for
 *           M <= 16, the single-CTA tcgen05 kernel's token warps above); fp16
 *           codes for M > 128 take the CTA-pair prefill kernel, which reads
 *           them directly and is the fastest path at prefill sizes
 *   qw      int8 [N, K] from ot_fold_weights, |qw| <= qmax(bits_w); 16-byte aligned
 *   sw, b_fold  fp32 [N]
 *   y_f16   fp16 [M, N], row stride ldy >= N
 *   workspace, workspace_bytes  optional device scratch (16-byte aligned) of
 *           at least ot_linear_workspace_size() bytes, ZERO-FILLED before its
 *           first use; the kernels keep it valid for every later call,
 *           including calls replayed from a CUDA graph (a launch counter in
 *           the workspace, not a value fixed at launch, tells one call's
 *           partial sums from another's).  With it,
 *           calls with M > 16 (tcgen05 kernels) and decode-sized calls (M <= 16) may
 *           share the (tile, K-slice) work evenly over the SMs and exchange
 *           exact int32 partial sums through it (stream-K); with NULL / too
 *           small, whole tiles are dealt out.  Calls that overlap on the GPU
 *           must not share a workspace.  The result is bit-identical either
 *           way.
 * Exactness: the tensor cores accumulate in fp32, which holds integers
 * exactly up to 2^24; the kernel therefore sums K in chunks short enough
 * that no partial sum can pass 2^24 for the promised bits, and adds the
 * chunks in int32.  Codes outside [-qmax, qmax] void that guarantee.
 * K * qmax_a * qmax_w must be < 2^31 (K <= 133144 for W8A8).
 */
ot_status ot_linear(const void *q, int q_format, int64_t M, int64_t K,
                    const int8_t *qw, const float *sw, const float *b_fold,
                    int64_t N, int bits_a, int bits_w, void *y_f16, int64_t ldy,
                    int relu, void *workspace, size_t workspace_bytes,
                    void *stream);

/*
 * ot_linear_workspace_size -- bytes of scratch that let ot_linear /
 * ot_linear_s32 balance prefill- and decode-sized calls over all SMs on the
 * current device (about 22.4 MB on a 152-SM GB300).  Host-only query.
 */
ot_status ot_linear_workspace_size(size_t *bytes);

/*
 * Per-token path (Eq. 3).  The paper quantizes the out and fc2 linears, whose
 * inputs carry no outlier channels, per token instead of per channel, and
 * carries the residual stream's symmetrization shift z in their bias (Eq. 8:
 * pass b + z as `bias`).
 *
 * ot_quantize_tokens -- dynamic symmetric quantization per token (Eq. 1 with
 * zero point 0, one scale per row):
 *   s_m = max_k |x[m,k]| / qmax_a,  q[m,k] = round_half_even(x[m,k] * qmax_a / max_k |x[m,k]|)
 * in fp32 (the reciprocal computed once per row); NaN is ignored by the max
 * and codes to 0; a row whose max is 0 or not finite gets s_m = 0, codes 0.
 *   x_f16  fp16 [M, K], row stride ldx (16-byte aligned; K, ldx % 8 == 0)
 *   q      [M, K] dense, int8 or fp16 codes (ot_code_format); 16-byte aligned
 *   s_tok  fp32 [M] out
 */
ot_status ot_quantize_tokens(const void *x_f16, int64_t M, int64_t K, int64_t ldx,
                             int bits_a, void *q, int q_format, float *s_tok,
                             void *stream);

/*
 * ot_quantize_weights -- per-output-channel symmetric weight codes with no
 * activation scale folded in (Eq. 3's W~):
 *   sw_n = max_k |W[n,k]| / qmax_w,  qw[n,k] = round(W[n,k] * qmax_w / max_k |W[n,k]|)
 *   w_f16 fp16 [N, K] (16-byte aligned, K % 16 == 0); qw int8 [N, K]; sw fp32 [N].
 */
ot_status ot_quantize_weights(const void *w_f16, int64_t N, int64_t K, int bits_w,
                              int8_t *qw, float *sw, void *stream);

/*
 * ot_linear_per_token -- Eq. 3 with the bias:
 *   y[m,n] = fp16( fma((float)acc[m,n], s_tok[m] * sw[n], bias[n]) ), ReLU if relu
 * with acc the exact integer product as in ot_linear; s_tok[m] * sw[n] is one
 * fp32 product.  Arguments as ot_linear plus s_tok fp32 [M] (from
 * ot_quantize_tokens) and bias fp32 [N] (b, or b + z for Eq. 8).
 */
ot_status ot_linear_per_token(const void *q_f16, int64_t M, int64_t K, const int8_t *qw,
                              const float *sw, const float *s_tok, const float *bias,
                              int64_t N, int bits_a, int bits_w, void *y_f16, int64_t ldy,
                              int relu, void *workspace, size_t workspace_bytes,
                              void *stream);

/*
 * ot_calibrate_clipped -- token-wise clipping calibration for models whose
 * linears have no bias (Appendix D: Llama cannot be symmetrized, and its
 * static activation scales are calibrated with token-wise clipping).  Per
 * channel k of X_cal [T, K] (fp16, row stride ldx), with T' the non-NaN
 * values and rho = ceil(alpha * T') evaluated in fp64:
 *   ch_hi[k] = the value of ascending rank rho,
 *   ch_lo[k] = the value of ascending rank T' + 1 - rho
 * (fp16 ordered by value, -0 before +0; alpha = 1 gives the min / max of
 * ot_calibrate).  A channel without non-NaN values gets lo = +inf, hi = -inf.
 * The whole calibration set is one call (order statistics do not accumulate
 * batch by batch); pass the range to ot_derive_params / ot_fold_weights as
 * ch_min / ch_max (symmetrize = 0 for bias-free models).
 *   alpha    in (0, 1], e.g. 0.999 to drop the 0.1 % most extreme tokens per side
 *   ch_lo, ch_hi  fp32 [K] out
 */
ot_status ot_calibrate_clipped(const void *x_f16, int64_t T, int64_t K, int64_t ldx,
                               double alpha, float *ch_lo, float *ch_hi, void *stream);

/*
 * LayerNorm fused with the symmetrization and the per-channel quantization
 * (Section 3.2: the codes of Eq. 7 come out of the LayerNorm before the linear,
 * whose gamma and beta absorb the scale r and the shift z).  For the linears
 * that follow a LayerNorm, h is the residual-stream input of that LayerNorm.
 *
 * ot_fold_layernorm -- offline, after calibration (z, r from ot_derive_params
 * or ot_fold_weights on the LayerNorm's outputs):
 *   gamma_r[k] = gamma[k] * r[k],   beta_r[k] = (beta[k] - z[k]) * r[k]   (fp32)
 *   gamma_f16, beta_f16  fp16 [K] (the LayerNorm's affine parameters)
 */
ot_status ot_fold_layernorm(const void *gamma_f16, const void *beta_f16, const float *z,
                            const float *r, int64_t K, float *gamma_r, float *beta_r,
                            void *stream);

/*
 * ot_layernorm_quantize -- codes of the symmetrized LayerNorm output:
 *   mean = sum_k h / K,  var = sum_k h^2 / K - mean^2 (biased),
 *   q[m,k] = round_half_even( ((h - mean) * rstd) * gamma_r[k] + beta_r[k] )
 * clipped to [-qmax, qmax], with rstd = 1 / sqrt(var + eps).  The statistics are
 * exact: h * 2^24 is an integer for every fp16 h, its sum S1 and the sum of
 * its squares S2 are exact integers, mean and rstd are formed from them by a
 * fixed sequence of IEEE fp32 operations (mean = (float(S1) / K) * 2^-24,
 * var = (float(K S2 - S1^2) / K / K) * 2^-48 with the 128-bit integer taken
 * as float(hi) 2^64 + float(lo), rstd = 1 / sqrt(var + eps)), then
 * (h - mean) * rstd and one fp32 fma, so the codes do not depend on the order
 * of any reduction.  A row holding a non-finite value codes to 0 throughout.
 *   h_f16   fp16 [M, K], row stride ldh (16-byte aligned; K, ldh % 8 == 0; K <= 2^22)
 *   gamma_r, beta_r  fp32 [K] from ot_fold_layernorm (16-byte aligned)
 *   eps     finite, >= 0
 *   q       [M, K] dense codes, int8 or fp16 (ot_code_format), 16-byte aligned
 *   rowsum  optional int32 [M]: sum_k q[m,k] (for ot_linear_asym), or NULL
 */
ot_status ot_layernorm_quantize(const void *h_f16, int64_t M, int64_t K, int64_t ldh,
                                const float *gamma_r, const float *beta_r, float eps,
                                int bits_a, void *q, int q_format, int32_t *rowsum,
                                void *stream);

/*
 * Asymmetric per-output-channel weights: the paper's "Int8" (Section 4,
 * Appendix A: zero points for the weights, min-max calibration), which trades
 * a little speed for accuracy against the symmetric "Int8*" of ot_fold_weights.
 *
 * ot_fold_weights_asym -- as ot_fold_weights (Eq. 5 fold, Eq. 7 bias), but each
 * row of W_s = W (.) s is quantized with Eq. 1 and a zero point over the range
 * [lo, hi] = [min(0, min_k W_s), max(0, max_k W_s)]:
 *   sw_n = (hi - lo) / (2^b - 1),  rw_n = (2^b - 1) / (hi - lo)
 *   zp_n = clip(round(-lo * rw_n), 0, 2^b - 1)
 *   u = clip(round(W_s * rw_n) + zp_n, 0, 2^b - 1),   W_s ~ (u - zp_n) sw_n
 * stored shifted so the codes fit int8:  qw = u - 2^(b-1),  zc_n = zp_n - 2^(b-1).
 * A row whose range is 0 or not finite gets sw = 0 and codes equal to zc.
 * Arguments as ot_fold_weights plus zc int32 [N] out (4-byte aligned).
 */
ot_status ot_fold_weights_asym(const float *ch_min, const float *ch_max, int bits_a,
                               int symmetrize, const void *w_f16, const void *b_f16,
                               int64_t N, int64_t K, int bits_w, float *z, float *s,
                               float *r, int8_t *qw, float *sw, int32_t *zc,
                               float *b_fold, void *stream);

/*
 * ot_quantize_act_rowsum -- ot_quantize_act plus the sum of each row's codes,
 *   rowsum[m] = sum_k q[m,k]   (int32 [M], exact; 4-byte aligned),
 * which the asymmetric-weight epilogue needs.  rowsum is cleared on `stream`
 * before the codes are added (integer atomics, so the result is exact and
 * independent of order).  K * qmax(bits_a) must be < 2^31.
 */
ot_status ot_quantize_act_rowsum(const void *x_f16, int64_t M, int64_t K, int64_t ldx,
                                 const float *z, const float *r, int bits_a, void *q,
                                 int q_format, int32_t *rowsum, void *stream);

/*
 * ot_linear_asym -- the quantized linear with asymmetric weights:
 *   acc[m,n] = sum_k q[m,k] * qw[n,k]                       exact integer
 *   y[m,n]   = fp16( fma((float)(acc[m,n] - zc_n * rowsum[m]), sw_n, b'_n) )
 where acc - zc_n * rowsum_m = sum_k q[m,k] (qw[n,k] - zc_n) is formed exactly
 * in integers and rounded once to fp32; ReLU before the fp16 rounding.
 * Arguments as ot_linear plus zc int32 [N] (from ot_fold_weights_asym) and
 * rowsum int32 [M] (from ot_quantize_act_rowsum).  |qw - zc| reaches
 * 2^bits_w - 1, so K * qmax(bits_a) * (2^bits_w - 1) must be < 2^31 (K <= 66,313
 * for W8A8; OT_ERR_UNSUPPORTED beyond).
 */
ot_status ot_linear_asym(const void *q_f16, int64_t M, int64_t K, const int8_t *qw,
                         const float *sw, const int32_t *zc, const int32_t *rowsum,
                         const float *b_fold, int64_t N, int bits_a, int bits_w,
                         void *y_f16, int64_t ldy, int relu, void *workspace,
                         size_t workspace_bytes, void *stream);

/* How ot_linear_fused joins the activation quantization to the product. */
typedef enum {
    OT_FUSE_AUTO = 0,      /* the faster form for the call (measured on GB300:
                              OT_FUSE_PDL at every token count) */
    OT_FUSE_PRODUCER = 1,  /* the linear's token producer quantizes X itself
                              (M <= 128 only) */
    OT_FUSE_PDL = 2        /* the quantize kernel writes the codes, the linear
                              runs as its programmatic dependent */
} ot_fuse_mode;

/*
 * ot_linear_fused -- the per-channel quantization of X (Eq. 6-7) and the
 * linear in one call: q = codes of X, y = fp16(fma(sum_k q qw, sw_n, b'_n)),
 * ReLU if relu; the result is bit-identical to ot_quantize_act followed by
 * ot_linear, in either form:
 *   - OT_FUSE_PDL: the quantize kernel writes the codes to q_f16 and the
 *     linear is launched as its programmatic dependent, so the linear's
 *     weight loads and set-up overlap the quantization and only its reads of
 *     the codes wait for it.
 *   - OT_FUSE_PRODUCER (M <= 128): the linear's own token producer reads fp16
 *     X with z and r and quantizes each tile in shared memory before the
 *     tensor cores read it (the quantization inside the GEMM's operand
 *     producer; one kernel, q_f16 not written).  Each token tile is then
 *     quantized once per weight tile instead of once in all, which on GB300
 *     costs more than the HBM round trip of the codes it saves.
 * x_f16 fp16 [M, ldx] (ldx >= K, ldx % 8 == 0, 16-byte aligned); z, r fp32 [K]
 * (16-byte aligned); q_f16: caller scratch fp16 [M, K], dense, 16-byte
 * aligned, whose contents are unspecified afterwards; mode an ot_fuse_mode
 * (OT_ERR_UNSUPPORTED for OT_FUSE_PRODUCER with M > 128); the remaining
 * arguments as ot_linear.  Same validation and errors as the two calls;
 * M == 0 launches nothing.
 */
ot_status ot_linear_fused(const void *x_f16, int64_t M, int64_t K, int64_t ldx, const float *z,
                          const float *r, int bits_a, const int8_t *qw, const float *sw,
                          const float *b_fold, int64_t N, int bits_w, void *q_f16, void *y_f16,
                          int64_t ldy, int relu, int mode, void *workspace,
                          size_t workspace_bytes, void *stream);

/*
 * ot_linear_quantize_next -- a linear whose output is the input of the next
 * per-channel quantized linear (fc1 -> ReLU -> fc2), with that layer's
 * activation quantization done in this epilogue (Section 3.2 fuses the
 * quantization into the producing kernel):
 *   v = fma((float)acc[m,n], sw_n, b'_n), then ReLU if relu,
 *   q_next[m,n] = round_half_even((v - z_next[n]) * r_next[n]) in [-qmax', qmax']
 * written as fp16 integers [M, ldq] -- the codes ot_linear takes as q_f16 for
 * the next layer, whose K is this layer's N.  The fp16 rounding of y is
 * skipped, so codes can differ by one from quantizing the fp16 y at a tie.
 * Arguments as ot_linear; z_next, r_next fp32 [N] (the next layer's z, r);
 * bits_next in [2, 8].  Symmetric weights only.
 */
ot_status ot_linear_quantize_next(const void *q_f16, int64_t M, int64_t K, const int8_t *qw,
                                  const float *sw, const float *b_fold, int64_t N, int bits_a,
                                  int bits_w, int relu, const float *z_next,
                                  const float *r_next, int bits_next, void *q_next_f16,
                                  int64_t ldq, void *workspace, size_t workspace_bytes,
                                  void *stream);

/*
 * ot_linear_noalloc -- ot_linear for callers that cannot allocate device
 * memory: for example a server or plugin that owns all GPU memory through
 * its own pool and forbids further cudaMalloc calls, or code that must not
 * risk an allocation failing (or synchronizing the device) in the middle of
 * a run.  The paper has no counterpart.  Same arguments and result as
 * ot_linear without the workspace: the stream-K scratch it would take is a
 * fixed 24 MiB array inside the library (a static device array that every
 * GPU loading the library holds until the process exits).  Nothing here
 * calls cudaMalloc, cudaFree or any allocating routine.
 *   - The first call on a device looks up the array's device address,
 *     zero-fills it on `stream` and waits for that fill (it synchronizes
 *     `stream` once); make that first call before any stream capture.  Later
 *     calls, from any thread or stream, find the array already cleared.
 *   - Every call shares the array and it keeps the last call's contents, so
 *     calls that overlap on the GPU (on different streams, or from several
 *     threads) race and may corrupt each other's results: serialize them.
 *   - Returns OT_ERR_UNSUPPORTED if the device would need more scratch than
 *     the array holds (more than 170 SMs; a 152-SM GB300 needs ~22.4 MB).
 */
ot_status ot_linear_noalloc(const void *q_f16, int64_t M, int64_t K,
                            const int8_t *qw, const float *sw,
                            const float *b_fold, int64_t N, int bits_a,
                            int bits_w, void *y_f16, int64_t ldy, int relu,
                            void *stream);

/*
 * ot_linear_s32 -- the same integer product as ot_linear, written out as the
 * int32 accumulators acc[m,n] (dense [M, N]) instead of the scaled fp16
 * output; the accumulators of Eq. 6 before external scaling, for checking.
 * q and q_format as in ot_linear.
 */
ot_status ot_linear_s32(const void *q, int q_format, int64_t M, int64_t K,
                        const int8_t *qw, int64_t N, int bits_a, int bits_w,
                        int32_t *acc, void *workspace, size_t workspace_bytes,
                        void *stream);

/*
 * ot_get_device_status -- synchronize `stream`, then return and clear the
 * device status word of the current device: OT_ERR_TIMEOUT if a bounded
 * device wait gave up since the last call; in a debug build OT_ERR_BOUNDS if
 * an index check failed since the last call; else OT_OK (or OT_ERR_CUDA if
 * the synchronization itself failed).
 */
ot_status ot_get_device_status(void *stream);

/*
 * ot_selftest_wait_timeout -- exercise the failure path of the bounded device
 * waits: one GPU thread waits on a barrier that nothing signals, gives up
 * after limit_ns (1 ms ... 2 s) and records OT_ERR_TIMEOUT in the device
 * status word, exactly as a stalled GEMM pipeline would; the kernel then
 * returns normally and the context stays usable.  The paper has no
 * counterpart; it exists so tests can check ot_get_device_status without
 * faulting or hanging a GPU.
 */
ot_status ot_selftest_wait_timeout(int64_t limit_ns, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* OUTLIERTUNE_H */
