/*
 * ot_oracle.c -- plain CPU oracle of the OutlierTune per-channel quantized
 * linear layer (arXiv 2406.18832).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call this file:
 * it is used by the tests, by __graft_entry__.smoke() and by the cpu_baseline
 * leg of bench.py.  It shares no code, header, table or constant with the CUDA
 * library; its only inputs are the raw arrays the tests generate.
 *
 * The method is an approximation (a quantizer), so this file takes the
 * algorithm's steps in the paper's order and notation, written plainly:
 *
 *   1. calibration: per-channel min / max over calibration tokens
 *      (Appendix A "min-max calibration"; Section 3.2 uses max/min per channel)
 *   2. symmetrization factor z_k = (max X[:,k] + min X[:,k]) / 2 and the static
 *      per-channel scale s_k of the symmetrized range (Section 3.2, Eq. 1 with
 *      z = 0, i.e. symmetric)
 *   3. pre-execution of dequantization: W_s = W (.) s^X (Eq. 5), per-output-
 *      channel quantization of W_s (Eq. 6 right-hand side) and the bias fold
 *      b' = b + z W^T (Eq. 7)
 *   4. per-channel activation quantization round(X_hat / s^X) (Eq. 6 / Eq. 7)
 *   5. the integer matrix product sum_k X~_ik (W~_s)_kj (Eq. 6)
 *   6. external scaling by s^{W_s}_j and the folded bias (Eq. 6, Eq. 7)
 *
 * Readings where the paper is silent (each is stated where it is used):
 *   R1 rounding  round() is round-half-to-even, evaluated in fp32.
 *   R2 division  X_hat / s is evaluated as X_hat * r with r = qmax / amp
 *                computed once per channel (fp32), likewise for the weights.
 *   R3 range     symmetric codes are restricted to [-qmax, qmax],
 *                qmax = 2^(bits-1) - 1; out-of-range values saturate.
 *   R4 scale     amp_k = max(max_k - z_k, z_k - min_k), s_k = amp_k / qmax.
 *   R5 degenerate a channel with amp = 0 (or no finite data) gets s = r = 0
 *                (codes 0); a weight row with amax = 0 gets sw = 0, codes 0.
 *   R6 non-finite NaN codes to 0; +-inf saturates to +-qmax.  Calibration
 *                ignores NaN.
 *   R7 bias      b' is formed in fp64 (k ascending) and rounded once to fp32.
 *   R8 epilogue  y = fp16( fma((float)acc, sw, b') ): the accumulator is
 *                rounded to fp32, the external scaling and bias take one
 *                fp32 fused multiply-add (one rounding), the result is
 *                rounded once to fp16 (half to even, overflow to +-inf);
 *                optional ReLU before the fp16 rounding.
 *   R9 Int8      the asymmetric weights ("Int8", Section 4 / Appendix A:
 *                zero points for the weights, min-max calibration) apply
 *                Eq. 1 to each row of W_s over the range [min(0, min),
 *                max(0, max)] (so 0 is exactly representable), with
 *                s = range / (2^b - 1), zero point round(-min * r) and codes
 *                clip(round(w * r) + zp, 0, 2^b - 1); NaN codes to the zero
 *                point.  Codes and zero points are stored shifted by
 *                -2^(b-1) so they fit int8.
 *   R10 LN fusion the paper fuses the per-channel quantization into the
 *                LayerNorm before the linear (Section 3.2) without fixing the
 *                arithmetic.  Here the row statistics are exact: h * 2^24 is
 *                an integer for every fp16 h, so sum(h) and sum(h^2) are
 *                exact integer sums; mean and 1/sqrt(var + eps) (biased
 *                variance) follow by a fixed sequence of IEEE fp32
 *                operations, and the codes by one fp32 fma with the folded
 *                gamma * r and (beta - z) * r.  A row holding a non-finite
 *                value codes to 0 throughout.
 *   R11 clipping the token-wise clipping the paper applies to bias-free
 *                models (Appendix D, after Outlier Suppression) replaces each
 *                channel's calibration min / max by order statistics over
 *                the calibration tokens: with T' the non-NaN values of the
 *                channel and rho = ceil(alpha * T') (fp64), the upper end is
 *                the value of ascending rank rho and the lower end the value
 *                of ascending rank T' + 1 - rho (alpha = 1: max and min).
 *                fp16 values are ordered by value with -0 before +0.
 *   R12 chaining when a linear's output feeds the next per-channel
 *                quantized linear (fc1 -> ReLU -> fc2, Section 3.2's fusion
 *                carried to the fc1 epilogue), the epilogue can write the
 *                next layer's codes directly: the fp32 value v of R8 (after
 *                ReLU) is quantized as round((v - z') * r') with the next
 *                layer's z', r' (R1-R3, R6); the fp16 rounding of y is
 *                skipped.
 *
 * Floating point: compile with -ffp-contract=off and no fast-math, so every
 * fp32 expression below rounds once per operation as written.
 */
#include <stdint.h>
#include <stddef.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------------------
 * IEEE 754 binary16 <-> binary32 / binary64, written from the format
 * definition: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits.
 * ------------------------------------------------------------------------- */
float ot_half_to_float(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 0x1f;
    int f = h & 0x3ff;
    double v;
    if (e == 0x1f)
        v = f ? NAN : INFINITY;
    else if (e == 0)
        v = ldexp((double)f, -24);             /* subnormal: f * 2^-14 * 2^-10 */
    else
        v = ldexp((double)(f + 1024), e - 25); /* (1 + f/1024) * 2^(e-15) */
    return (float)(sign ? -v : v);             /* exact: 11 bits fit in fp32 */
}

/* Round-half-to-even of a finite double to binary16; overflow gives +-inf. */
uint16_t ot_double_to_half(double v)
{
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (isnan(v)) return 0x7e00;
    if (isinf(v)) return sign | 0x7c00;
    /* binary16 numbers are n * 2^q with integer n < 2048; q = -24 for the
       subnormal / smallest normal binade, q = e - 10 for the binade [2^e, 2^(e+1)). */
    int e;
    frexp(a, &e);            /* a = m * 2^e, m in [0.5, 1): a in [2^(e-1), 2^e) */
    int q = (e - 1) - 10;
    if (q < -24) q = -24;
    double n = ldexp(a, -q); /* exact: scaling by a power of two */
    double n_int = nearbyint(n); /* default rounding mode: half to even */
    if (n_int >= 2048.0) {   /* rounded up into the next binade */
        n_int /= 2.0;
        q += 1;
    }
    if (q > 15 - 10 || (q == 5 && n_int >= 2048.0)) return sign | 0x7c00;
    uint16_t bits;
    if (n_int < 1024.0) {    /* subnormal (q == -24) */
        bits = (uint16_t)n_int;
    } else {
        int exp_field = q + 10 + 15; /* n in [1024, 2048): value = (n/1024) * 2^(q+10) */
        bits = (uint16_t)((exp_field << 10) | ((int)n_int - 1024));
    }
    return sign | bits;
}

static int qmax_of(int bits) { return (1 << (bits - 1)) - 1; }

/* Round half to even in fp32, then saturate to [-qmax, qmax] (R1, R3, R6). */
static int quantize_code(float u, int qmax)
{
    if (isnan(u)) return 0;
    if (u >= (float)qmax) return qmax;
    if (u <= -(float)qmax) return -qmax;
    return (int)nearbyintf(u);
}

/* ---------------------------------------------------------------------------
 * Step 1: calibration (Appendix A, Section 3.2).  Running per-channel min and
 * max of X_cal[T, K] (fp16, row stride ldx elements).  reset = 1 starts from
 * (+inf, -inf); reset = 0 continues from the values already in mn / mx, so a
 * calibration set can be fed batch by batch.
 * ------------------------------------------------------------------------- */
void oracle_calibrate(const uint16_t *x, int64_t T, int64_t K, int64_t ldx,
                      float *mn, float *mx, int reset)
{
    if (reset)
        for (int64_t k = 0; k < K; ++k) { mn[k] = INFINITY; mx[k] = -INFINITY; }
    for (int64_t t = 0; t < T; ++t)
        for (int64_t k = 0; k < K; ++k) {
            float v = ot_half_to_float(x[t * ldx + k]);
            if (isnan(v)) continue;          /* R6 */
            if (v < mn[k]) mn[k] = v;
            if (v > mx[k]) mx[k] = v;
        }
}

/* ---------------------------------------------------------------------------
 * Step 2: symmetrization factor and static scale (Section 3.2; Eq. 1, z = 0).
 *   z_k   = (max_k + min_k) / 2
 *   amp_k = max(max_k - z_k, z_k - min_k)                              (R4)
 *   s_k   = amp_k / qmax,   r_k = qmax / amp_k                         (R2)
 * With symmetrize = 0 (the "Non-Sym" ablation of Table 6) z_k = 0 and
 * amp_k = max(|max_k|, |min_k|).
 * ------------------------------------------------------------------------- */
void oracle_params(const float *mn, const float *mx, int64_t K, int bits,
                   int symmetrize, float *z, float *s, float *r)
{
    const float qmax = (float)qmax_of(bits);
    for (int64_t k = 0; k < K; ++k) {
        float lo = mn[k], hi = mx[k];
        float zk, amp;
        if (!(lo <= hi) || isinf(lo) || isinf(hi)) {    /* no finite data (R5) */
            z[k] = 0.0f; s[k] = 0.0f; r[k] = 0.0f;
            continue;
        }
        if (symmetrize) {
            zk = (hi + lo) * 0.5f;
            float up = hi - zk, down = zk - lo;
            amp = up > down ? up : down;
        } else {
            zk = 0.0f;
            float a = fabsf(hi), b = fabsf(lo);
            amp = a > b ? a : b;
        }
        z[k] = zk;
        if (amp > 0.0f && isfinite(amp)) {
            s[k] = amp / qmax;
            r[k] = qmax / amp;
        } else {
            s[k] = 0.0f; r[k] = 0.0f;
        }
    }
}

/* ---------------------------------------------------------------------------
 * Step 3: pre-execution of dequantization and bias correction.
 *   W_s[n,k] = W[n,k] * s_k                         (Eq. 5, W is [N, K])
 *   amax_n   = max_k |W_s[n,k]|
 *   sw_n     = amax_n / qmax_w,  rw_n = qmax_w / amax_n              (R2, R5)
 *   qw[n,k]  = round(W_s[n,k] * rw_n) in [-qmax_w, qmax_w]   (Eq. 6 right side)
 *   b'_n     = b_n + sum_k z_k W[n,k]                      (Eq. 7, R7)
 * b may be NULL (no bias).
 * ------------------------------------------------------------------------- */
void oracle_fold(const uint16_t *w, const uint16_t *b, int64_t N, int64_t K,
                 const float *z, const float *s, int bits_w,
                 int8_t *qw, float *sw, float *bfold)
{
    const int qmax = qmax_of(bits_w);
    for (int64_t n = 0; n < N; ++n) {
        const uint16_t *wrow = w + n * K;
        float amax = 0.0f;
        for (int64_t k = 0; k < K; ++k) {
            float ws = ot_half_to_float(wrow[k]) * s[k];
            float a = fabsf(ws);
            if (a > amax) amax = a;
        }
        float swn = 0.0f, rwn = 0.0f;
        if (amax > 0.0f && isfinite(amax)) {
            swn = amax / (float)qmax;
            rwn = (float)qmax / amax;
        }
        sw[n] = swn;
        for (int64_t k = 0; k < K; ++k) {
            float ws = ot_half_to_float(wrow[k]) * s[k];
            qw[n * K + k] = (int8_t)quantize_code(ws * rwn, qmax);
        }
        double acc = b ? (double)ot_half_to_float(b[n]) : 0.0;
        for (int64_t k = 0; k < K; ++k)
            acc += (double)z[k] * (double)ot_half_to_float(wrow[k]);
        bfold[n] = (float)acc;
    }
}

/* ---------------------------------------------------------------------------
 * Step 4: per-channel static activation quantization, round(X_hat / s^X) with
 * X_hat = X - z (Eq. 6, Eq. 7; R1-R3, R6):
 *   t = x - z_k (fp32),  u = t * r_k (fp32),  q = round_half_even(u) saturated.
 * X is [M, K] fp16 with row stride ldx; q is [M, K] int8, dense.
 * ------------------------------------------------------------------------- */
void oracle_quantize(const uint16_t *x, int64_t M, int64_t K, int64_t ldx,
                     const float *z, const float *r, int bits_a, int8_t *q)
{
    const int qmax = qmax_of(bits_a);
    for (int64_t m = 0; m < M; ++m)
        for (int64_t k = 0; k < K; ++k) {
            float t = ot_half_to_float(x[m * ldx + k]) - z[k];
            float u = t * r[k];
            q[m * K + k] = (int8_t)quantize_code(u, qmax);
        }
}

/* ---------------------------------------------------------------------------
 * Step 5: the integer product of Eq. 6, acc[m,n] = sum_k q[m,k] * qw[n,k],
 * in int64 (the caller checks that it fits the int32 accumulator).
 * ------------------------------------------------------------------------- */
void oracle_matmul(const int8_t *q, const int8_t *qw, int64_t M, int64_t N,
                   int64_t K, int64_t *acc)
{
    for (int64_t m = 0; m < M; ++m)
        for (int64_t n = 0; n < N; ++n) {
            int64_t sum = 0;
            for (int64_t k = 0; k < K; ++k)
                sum += (int64_t)q[m * K + k] * (int64_t)qw[n * K + k];
            acc[m * N + n] = sum;
        }
}

/* ---------------------------------------------------------------------------
 * Step 6: external scaling (Eq. 6) plus the folded bias (Eq. 7), R8:
 *   y[m,n] = fp16( fma((float)acc[m,n], sw_n, b'_n) ),  ReLU applied before
 * the fp16 rounding when relu != 0.  y holds binary16 bit patterns.
 * ------------------------------------------------------------------------- */
void oracle_epilogue(const int64_t *acc, int64_t M, int64_t N, const float *sw,
                     const float *bfold, int relu, uint16_t *y)
{
    for (int64_t m = 0; m < M; ++m)
        for (int64_t n = 0; n < N; ++n) {
            float a = (float)acc[m * N + n];       /* round to nearest even */
            float v = fmaf(a, sw[n], bfold[n]);    /* one rounding */
            if (relu && !(v > 0.0f)) v = 0.0f;
            y[m * N + n] = ot_double_to_half((double)v);
        }
}

/* ---------------------------------------------------------------------------
 * Per-token path (Eq. 3; used by the paper for the out and fc2 linears,
 * whose inputs carry no outlier channels, with Eq. 8 folding the residual
 * stream's symmetrization shift into their bias).
 *
 * Step T1: dynamic symmetric quantization per token (Eq. 1 with z = 0, one
 * scale per row of X):
 *   amax_m = max_k |x[m,k]|  (NaN ignored),
 *   s_m = amax_m / qmax, r_m = qmax / amax_m  (fp32; both 0 when amax_m is 0
 *   or not finite), q[m,k] = round_half_even(x[m,k] * r_m) in [-qmax, qmax].
 * ------------------------------------------------------------------------- */
void oracle_quantize_tokens(const uint16_t *x, int64_t M, int64_t K, int64_t ldx,
                            int bits, int8_t *q, float *s_tok)
{
    const int qmax = qmax_of(bits);
    for (int64_t m = 0; m < M; ++m) {
        float amax = 0.0f;
        for (int64_t k = 0; k < K; ++k) {
            float a = fabsf(ot_half_to_float(x[m * ldx + k]));
            if (a > amax) amax = a;          /* NaN compares false: ignored */
        }
        float s = 0.0f, r = 0.0f;
        if (amax > 0.0f && isfinite(amax)) {
            s = amax / (float)qmax;
            r = (float)qmax / amax;
        }
        s_tok[m] = s;
        for (int64_t k = 0; k < K; ++k)
            q[m * K + k] = (int8_t)quantize_code(ot_half_to_float(x[m * ldx + k]) * r, qmax);
    }
}

/* ---------------------------------------------------------------------------
 * Step T3: external scaling of Eq. 3 by the token scale and the output-channel
 * scale, plus the bias:
 *   y[m,n] = fp16( fma((float)acc[m,n], s_m * sw_n, b_n) )
 * where s_m * sw_n is one fp32 product; ReLU before the fp16 rounding.
 * (The weights of this path are quantized per output channel without any
 * activation scale: oracle_fold with s = 1, z = 0.)
 * ------------------------------------------------------------------------- */
void oracle_epilogue_tokens(const int64_t *acc, int64_t M, int64_t N, const float *s_tok,
                            const float *sw, const float *bias, int relu, uint16_t *y)
{
    for (int64_t m = 0; m < M; ++m)
        for (int64_t n = 0; n < N; ++n) {
            float a = (float)acc[m * N + n];
            float scale = s_tok[m] * sw[n];
            float v = fmaf(a, scale, bias[n]);
            if (relu && !(v > 0.0f)) v = 0.0f;
            y[m * N + n] = ot_double_to_half((double)v);
        }
}

/* ---------------------------------------------------------------------------
 * Asymmetric per-output-channel weights ("Int8", R9; Eq. 1 with z != 0).
 *
 * Step A3': Eq. 1 on each row of W_s = W (.) s^X (Eq. 5):
 *   lo_n = min(0, min_k W_s[n,k]),  hi_n = max(0, max_k W_s[n,k])
 *   sw_n = (hi_n - lo_n) / (2^b - 1),  rw_n = (2^b - 1) / (hi_n - lo_n)   (R2)
 *   zp_n = clip(round(-lo_n * rw_n), 0, 2^b - 1)
 *   u[n,k] = clip(round(W_s[n,k] * rw_n) + zp_n, 0, 2^b - 1)
 * so that W_s[n,k] ~ (u[n,k] - zp_n) * sw_n.  Stored shifted by -2^(b-1):
 *   qw[n,k] = u[n,k] - 2^(b-1),  zc_n = zp_n - 2^(b-1),  W_s ~ (qw - zc) sw.
 * A row whose range is 0 or not finite gets sw = 0 and every code equal to
 * its zero point (dequantizing to 0).  s may be NULL (s_k = 1).
 * ------------------------------------------------------------------------- */
static int asym_code(float u, int zp, int umax)
{
    int c;
    if (u != u) {
        c = 0;                                /* NaN: the zero point */
    } else {
        float r = nearbyintf(u);              /* R1 */
        if (r > (float)umax) c = umax;        /* the clip below decides */
        else if (r < -(float)umax) c = -umax;
        else c = (int)r;
    }
    c += zp;
    return c < 0 ? 0 : (c > umax ? umax : c);
}

void oracle_fold_codes_asym(const uint16_t *w, int64_t N, int64_t K, const float *s,
                            int bits_w, int8_t *qw, float *sw, int32_t *zc)
{
    const int umax = (1 << bits_w) - 1;
    const int shift = 1 << (bits_w - 1);
    for (int64_t n = 0; n < N; ++n) {
        const uint16_t *wrow = w + n * K;
        float lo = 0.0f, hi = 0.0f;
        for (int64_t k = 0; k < K; ++k) {
            float ws = ot_half_to_float(wrow[k]) * (s ? s[k] : 1.0f);
            if (ws < lo) lo = ws;               /* NaN compares false */
            if (ws > hi) hi = ws;
        }
        float range = hi - lo;
        float swn = 0.0f, rwn = 0.0f;
        int zp = 0;
        if (range > 0.0f && isfinite(range)) {
            swn = range / (float)umax;
            rwn = (float)umax / range;
            zp = asym_code(-lo * rwn, 0, umax);
        }
        sw[n] = swn;
        zc[n] = zp - shift;
        for (int64_t k = 0; k < K; ++k) {
            float ws = ot_half_to_float(wrow[k]) * (s ? s[k] : 1.0f);
            qw[n * K + k] = (int8_t)(asym_code(ws * rwn, zp, umax) - shift);
        }
    }
}

/* Sum of each row's activation codes, rs[m] = sum_k q[m,k] (exact). */
void oracle_rowsum(const int8_t *q, int64_t M, int64_t K, int64_t *rs)
{
    for (int64_t m = 0; m < M; ++m) {
        int64_t t = 0;
        for (int64_t k = 0; k < K; ++k) t += q[m * K + k];
        rs[m] = t;
    }
}

/* ---------------------------------------------------------------------------
 * Step A6': external scaling with the weight zero point.  With
 * acc[m,n] = sum_k q[m,k] qw[n,k] (Eq. 6 on the stored codes),
 *   sum_k q[m,k] (qw[n,k] - zc_n) = acc[m,n] - zc_n * rs[m]   (exact, int64)
 *   y[m,n] = fp16( fma((float)(acc[m,n] - zc_n rs[m]), sw_n, b'_n) )
 * (R8 otherwise; ReLU before the fp16 rounding).
 * ------------------------------------------------------------------------- */
void oracle_epilogue_asym(const int64_t *acc, const int64_t *rs, const int32_t *zc,
                          int64_t M, int64_t N, const float *sw, const float *bfold,
                          int relu, uint16_t *y)
{
    for (int64_t m = 0; m < M; ++m)
        for (int64_t n = 0; n < N; ++n) {
            int64_t t = acc[m * N + n] - (int64_t)zc[n] * rs[m];
            float a = (float)t;                    /* round to nearest even */
            float v = fmaf(a, sw[n], bfold[n]);    /* one rounding */
            if (relu && !(v > 0.0f)) v = 0.0f;
            y[m * N + n] = ot_double_to_half((double)v);
        }
}

/* ---------------------------------------------------------------------------
 * LayerNorm fused with the symmetrization and the per-channel quantization
 * (Section 3.2, R10): LN(h) = (h - mean) / sqrt(var + eps) * gamma + beta, and
 * the codes round((LN(h) - z) * r) = round(n * gamma * r + (beta - z) * r)
 * with n = (h - mean) / sqrt(var + eps).
 *
 * Step L0 (offline, with the fold): gamma_r[k] = gamma[k] * r[k] and
 * beta_r[k] = (beta[k] - z[k]) * r[k] in fp32 (gamma, beta fp16).
 * ------------------------------------------------------------------------- */
void oracle_fold_layernorm(const uint16_t *gamma, const uint16_t *beta, const float *z,
                           const float *r, int64_t K, float *gamma_r, float *beta_r)
{
    for (int64_t k = 0; k < K; ++k) {
        gamma_r[k] = ot_half_to_float(gamma[k]) * r[k];
        beta_r[k] = (ot_half_to_float(beta[k]) - z[k]) * r[k];
    }
}

/* A non-negative 128-bit integer as hi * 2^64 + lo, each part converted to
 * float and added (round to nearest at each step; the scaling is exact). */
static float u128_to_float(unsigned __int128 v)
{
    const uint64_t hi = (uint64_t)(v >> 64), lo = (uint64_t)v;
    return (float)hi * 18446744073709551616.0f + (float)lo;
}

/* ---------------------------------------------------------------------------
 * Step L1: per row m of the hidden state h [M, K] (fp16, row stride ldh):
 *   H_k  = h_k * 2^24 (integer),  S1 = sum_k H_k,  S2 = sum_k H_k^2   (exact)
 *   mean = ((float)S1 / K) * 2^-24                              (fp32)
 *   V    = K * S2 - S1^2  (exact, >= 0),  var = (float(V) / K / K) * 2^-48
 *   rstd = 1 / sqrt(var + eps)                                   (fp32, IEEE)
 *   u_k  = fma((h_k - mean) * rstd, gamma_r[k], beta_r[k])   (fp32 roundings)
 *   q_k  = round_half_even(u_k) in [-qmax, qmax]
 * q is [M, K] int8; rowsum[m] = sum_k q[m,k] if rowsum is not NULL; mean and
 * rstd per row are returned for the tests (NULL to skip).
 * ------------------------------------------------------------------------- */
void oracle_layernorm_quantize(const uint16_t *h, int64_t M, int64_t K, int64_t ldh,
                               const float *gamma_r, const float *beta_r, float eps,
                               int bits, int8_t *q, int64_t *rowsum, float *mean_out,
                               float *rstd_out)
{
    const int qmax = qmax_of(bits);
    for (int64_t m = 0; m < M; ++m) {
        const uint16_t *row = h + m * ldh;
        int64_t s1 = 0;
        unsigned __int128 s2 = 0;
        int finite = 1;
        for (int64_t k = 0; k < K; ++k) {
            const float v = ot_half_to_float(row[k]);
            if (!isfinite(v)) { finite = 0; break; }
            const int64_t hk = (int64_t)(v * 16777216.0f);   /* exact: an fp16 times 2^24 */
            s1 += hk;
            const uint64_t a = (uint64_t)(hk < 0 ? -hk : hk);
            s2 += (unsigned __int128)a * a;
        }
        float mean = 0.0f, rstd = 0.0f;
        if (finite) {
            const float kf = (float)K;
            mean = ((float)s1 / kf) * 0x1p-24f;
            const __int128 s1s = (__int128)s1;
            const unsigned __int128 v = (unsigned __int128)K * s2 - (unsigned __int128)(s1s * s1s);
            const float var = ((u128_to_float(v) / kf) / kf) * 0x1p-48f;
            rstd = 1.0f / sqrtf(var + eps);
        }
        if (mean_out) mean_out[m] = mean;
        if (rstd_out) rstd_out[m] = rstd;
        int64_t rs = 0;
        for (int64_t k = 0; k < K; ++k) {
            int c = 0;
            if (finite) {
                const float n = (ot_half_to_float(row[k]) - mean) * rstd;
                c = quantize_code(fmaf(n, gamma_r[k], beta_r[k]), qmax);
            }
            q[m * K + k] = (int8_t)c;
            rs += c;
        }
        if (rowsum) rowsum[m] = rs;
    }
}

/* ---------------------------------------------------------------------------
 * Token-wise clipping calibration (R11; Appendix D): per channel k of
 * X_cal [T, K] (fp16, row stride ldx), the clipped range [lo_k, hi_k] at
 * quantile alpha in (0, 1].  A channel without non-NaN values gets
 * lo = +inf, hi = -inf (as min / max of nothing).
 * ------------------------------------------------------------------------- */
static uint16_t order_key(uint16_t h)       /* monotone in the fp16 value */
{
    return (h & 0x8000u) ? (uint16_t)~h : (uint16_t)(h | 0x8000u);
}

static int cmp_u16(const void *a, const void *b)
{
    const uint16_t x = *(const uint16_t *)a, y = *(const uint16_t *)b;
    return (x > y) - (x < y);
}

void oracle_calibrate_clipped(const uint16_t *x, int64_t T, int64_t K, int64_t ldx, double alpha,
                              float *lo, float *hi)
{
    uint16_t *keys = (uint16_t *)malloc((size_t)(T > 0 ? T : 1) * sizeof(uint16_t));
    for (int64_t k = 0; k < K; ++k) {
        int64_t n = 0;
        for (int64_t t = 0; t < T; ++t) {
            const uint16_t h = x[t * ldx + k];
            if ((h & 0x7C00u) == 0x7C00u && (h & 0x03FFu)) continue;   /* NaN */
            keys[n++] = order_key(h);
        }
        if (n == 0) {
            lo[k] = INFINITY;
            hi[k] = -INFINITY;
            continue;
        }
        qsort(keys, (size_t)n, sizeof(uint16_t), cmp_u16);
        int64_t rho = (int64_t)ceil(alpha * (double)n);
        if (rho < 1) rho = 1;
        if (rho > n) rho = n;
        const uint16_t kh = keys[rho - 1], kl = keys[n - rho];
        const uint16_t bh = (kh & 0x8000u) ? (uint16_t)(kh & 0x7FFFu) : (uint16_t)~kh;
        const uint16_t bl = (kl & 0x8000u) ? (uint16_t)(kl & 0x7FFFu) : (uint16_t)~kl;
        hi[k] = ot_half_to_float(bh);
        lo[k] = ot_half_to_float(bl);
    }
    free(keys);
}

/* ---------------------------------------------------------------------------
 * Step A6'' (R12): the epilogue of a linear whose output is the next linear's
 * input, writing that layer's codes instead of y:
 *   v = fma((float)acc[m,n], sw_n, b'_n),  ReLU if relu,
 *   q'[m,n] = round_half_even((v - z'_n) * r'_n) in [-qmax', qmax']   (fp32)
 * z', r' [N] are the next layer's symmetrization and reciprocal scale.
 * ------------------------------------------------------------------------- */
void oracle_epilogue_quantize(const int64_t *acc, int64_t M, int64_t N, const float *sw,
                              const float *bfold, int relu, const float *zn, const float *rn,
                              int bits_next, int8_t *q)
{
    const int qmax = qmax_of(bits_next);
    for (int64_t m = 0; m < M; ++m)
        for (int64_t n = 0; n < N; ++n) {
            float a = (float)acc[m * N + n];
            float v = fmaf(a, sw[n], bfold[n]);
            if (relu && !(v > 0.0f)) v = 0.0f;
            float t = v - zn[n];
            q[m * N + n] = (int8_t)quantize_code(t * rn[n], qmax);
        }
}
