// fold.cu -- pre-execution of dequantization (Eq. 5), per-output-channel
// weight quantization of W_s (Eq. 6 right-hand side) and the bias fold
// b' = b + z W^T (Eq. 7).  Offline, once per layer.
#include <cuda_fp16.h>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

OT_DEBUG_UNIT(fold)

namespace {

constexpr int kFoldThreads = 256;

// One CTA per output row n (grid-stride): amax_n = max_k |W[n,k] * s_k|, then
// sw_n, rw_n and the codes round(W[n,k] * s_k * rw_n).  s == null means s_k = 1
// (per-output-channel weight codes without activation scales, Eq. 3's W~).  Each thread handles
// 8 consecutive k per step (16-byte loads of W, 8-byte stores of codes).
__global__ void __launch_bounds__(kFoldThreads) fold_codes_kernel(const __half *__restrict__ w, int64_t N,
                                                                  int64_t K, const float *__restrict__ s,
                                                                  float qmax, int iqmax, int8_t *qw, float *sw) {
    __shared__ float red[kFoldThreads / 32];
    __shared__ float s_rw;
    for (int64_t n = blockIdx.x; n < N; n += gridDim.x) {
        const __half *row = w + n * K;
        float amax = 0.f;
        for (int64_t k = (int64_t)threadIdx.x * 8; k < K; k += kFoldThreads * 8) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(row + k));
            const __half2 *h = reinterpret_cast<const __half2 *>(&v);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __half22float2(h[j]);
                amax = fmaxf(amax, fabsf(__fmul_rn(f.x, (s ? __ldg(s + k + 2 * j) : 1.0f))));
                amax = fmaxf(amax, fabsf(__fmul_rn(f.y, (s ? __ldg(s + k + 2 * j + 1) : 1.0f))));
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
        __syncthreads();
        if (threadIdx.x == 0) {
            float a = red[0];
            for (int i = 1; i < kFoldThreads / 32; ++i) a = fmaxf(a, red[i]);
            float swn = 0.f, rwn = 0.f;
            if (a > 0.f && isfinite(a)) {
                swn = __fdiv_rn(a, qmax);
                rwn = __fdiv_rn(qmax, a);
            }
            sw[n] = swn;
            s_rw = rwn;
        }
        __syncthreads();
        const float rw = s_rw;
        for (int64_t k = (int64_t)threadIdx.x * 8; k < K; k += kFoldThreads * 8) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(row + k));
            const __half2 *h = reinterpret_cast<const __half2 *>(&v);
            uint32_t b[8];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __half22float2(h[j]);
                const int c0 = __float2int_rn(__fmul_rn(__fmul_rn(f.x, (s ? __ldg(s + k + 2 * j) : 1.0f)), rw));
                const int c1 = __float2int_rn(__fmul_rn(__fmul_rn(f.y, (s ? __ldg(s + k + 2 * j + 1) : 1.0f)), rw));
                b[2 * j] = (uint32_t)max(-iqmax, min(iqmax, c0));
                b[2 * j + 1] = (uint32_t)max(-iqmax, min(iqmax, c1));
            }
            uint2 o;
            o.x = __byte_perm(__byte_perm(b[0], b[1], 0x0040), __byte_perm(b[2], b[3], 0x0040), 0x5410);
            o.y = __byte_perm(__byte_perm(b[4], b[5], 0x0040), __byte_perm(b[6], b[7], 0x0040), 0x5410);
            if (OT_DCHECK(k + 8 <= K)) *reinterpret_cast<uint2 *>(qw + n * K + k) = o;
        }
        __syncthreads();
    }
}

// Asymmetric per-output-channel codes ("Int8" weights; Eq. 1 with a zero
// point): one CTA per row n (grid-stride) takes lo = min(0, min_k W_s[n,k])
// and hi = max(0, max_k W_s[n,k]) with W_s = W (.) s, then sw_n = (hi - lo) /
// (2^b - 1), rw_n = (2^b - 1) / (hi - lo), the zero point zp = clip(round(-lo *
// rw), 0, 2^b - 1) and the codes u = clip(round(W_s * rw) + zp, 0, 2^b - 1),
// stored as u - 2^(b-1) (zc_n = zp - 2^(b-1)).  A row whose range is 0 or not
// finite gets sw = 0 and every code equal to its zero point.  NaN codes to the
// zero point (cvt.rni gives 0).
__device__ __forceinline__ int asym_code(float u, int zp, int umax) {
    const int c = max(-umax, min(umax, __float2int_rn(u)));
    return max(0, min(umax, c + zp));
}

__global__ void __launch_bounds__(kFoldThreads) fold_codes_asym_kernel(const __half *__restrict__ w, int64_t N,
                                                                       int64_t K, const float *__restrict__ s,
                                                                       int umax, int8_t *qw, float *sw,
                                                                       int32_t *zc) {
    __shared__ float rlo[kFoldThreads / 32], rhi[kFoldThreads / 32];
    __shared__ float s_rw;
    __shared__ int s_zp;
    const int shift = (umax + 1) / 2;
    for (int64_t n = blockIdx.x; n < N; n += gridDim.x) {
        const __half *row = w + n * K;
        float lo = 0.f, hi = 0.f;
        for (int64_t k = (int64_t)threadIdx.x * 8; k < K; k += kFoldThreads * 8) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(row + k));
            const __half2 *h = reinterpret_cast<const __half2 *>(&v);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __half22float2(h[j]);
                const float a = __fmul_rn(f.x, s ? __ldg(s + k + 2 * j) : 1.0f);
                const float b = __fmul_rn(f.y, s ? __ldg(s + k + 2 * j + 1) : 1.0f);
                lo = fminf(lo, fminf(a, b));  // fminf ignores NaN
                hi = fmaxf(hi, fmaxf(a, b));
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
            hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
        }
        if ((threadIdx.x & 31) == 0) {
            rlo[threadIdx.x >> 5] = lo;
            rhi[threadIdx.x >> 5] = hi;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            float l = rlo[0], h = rhi[0];
            for (int i = 1; i < kFoldThreads / 32; ++i) {
                l = fminf(l, rlo[i]);
                h = fmaxf(h, rhi[i]);
            }
            const float range = __fsub_rn(h, l);
            float swn = 0.f, rwn = 0.f;
            int zp = 0;
            if (range > 0.f && isfinite(range)) {
                swn = __fdiv_rn(range, (float)umax);
                rwn = __fdiv_rn((float)umax, range);
                zp = asym_code(__fmul_rn(-l, rwn), 0, umax);
            }
            sw[n] = swn;
            zc[n] = zp - shift;
            s_rw = rwn;
            s_zp = zp;
        }
        __syncthreads();
        const float rw = s_rw;
        const int zp = s_zp;
        for (int64_t k = (int64_t)threadIdx.x * 8; k < K; k += kFoldThreads * 8) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(row + k));
            const __half2 *h = reinterpret_cast<const __half2 *>(&v);
            uint32_t b[8];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __half22float2(h[j]);
                const float a0 = __fmul_rn(f.x, s ? __ldg(s + k + 2 * j) : 1.0f);
                const float a1 = __fmul_rn(f.y, s ? __ldg(s + k + 2 * j + 1) : 1.0f);
                b[2 * j] = (uint32_t)(asym_code(__fmul_rn(a0, rw), zp, umax) - shift);
                b[2 * j + 1] = (uint32_t)(asym_code(__fmul_rn(a1, rw), zp, umax) - shift);
            }
            uint2 o;
            o.x = __byte_perm(__byte_perm(b[0], b[1], 0x0040), __byte_perm(b[2], b[3], 0x0040), 0x5410);
            o.y = __byte_perm(__byte_perm(b[4], b[5], 0x0040), __byte_perm(b[6], b[7], 0x0040), 0x5410);
            if (OT_DCHECK(k + 8 <= K)) *reinterpret_cast<uint2 *>(qw + n * K + k) = o;
        }
        __syncthreads();
    }
}

// b'_n = b_n + sum_k z_k W[n,k]: one thread per row, k ascending, in fp64.
// Each product of an fp32 and an fp16 value is exact in fp64, so the only
// roundings are those of the running sum, taken in the same order as a plain
// sequential loop, and the final rounding to fp32.
__global__ void __launch_bounds__(128) fold_bias_kernel(const __half *__restrict__ w, const __half *__restrict__ b,
                                                        int64_t N, int64_t K, const float *__restrict__ z,
                                                        float *bfold) {
    const int64_t n = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (n >= N) return;
    const __half *row = w + n * K;
    double acc = b ? (double)__half2float(b[n]) : 0.0;
    for (int64_t k = 0; k < K; k += 8) {
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(row + k));
        const __half *h = reinterpret_cast<const __half *>(&v);
#pragma unroll
        for (int j = 0; j < 8; ++j)
            acc = __dadd_rn(acc, __dmul_rn((double)__ldg(z + k + j), (double)__half2float(h[j])));
    }
    bfold[n] = __double2float_rn(acc);
}

}  // namespace

cudaError_t launch_fold(const void *w, const void *b, int64_t N, int64_t K, const float *z, const float *s,
                        int bits_w, int8_t *qw, float *sw, float *bfold, cudaStream_t st) {
    if (N == 0) return cudaSuccess;
    const int iqmax = (1 << (bits_w - 1)) - 1;
    const int64_t grid = N < 65535 * 4 ? N : 65535 * 4;
    fold_codes_kernel<<<(unsigned)grid, kFoldThreads, 0, st>>>(reinterpret_cast<const __half *>(w), N, K, s,
                                                               (float)iqmax, iqmax, qw, sw);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    fold_bias_kernel<<<(unsigned)((N + 127) / 128), 128, 0, st>>>(reinterpret_cast<const __half *>(w),
                                                                  reinterpret_cast<const __half *>(b), N, K, z,
                                                                  bfold);
    return cudaGetLastError();
}

cudaError_t launch_fold_asym(const void *w, const void *b, int64_t N, int64_t K, const float *z, const float *s,
                             int bits_w, int8_t *qw, float *sw, int32_t *zc, float *bfold, cudaStream_t st) {
    if (N == 0) return cudaSuccess;
    const int64_t grid = N < 65535 * 4 ? N : 65535 * 4;
    fold_codes_asym_kernel<<<(unsigned)grid, kFoldThreads, 0, st>>>(reinterpret_cast<const __half *>(w), N, K, s,
                                                                    (1 << bits_w) - 1, qw, sw, zc);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    fold_bias_kernel<<<(unsigned)((N + 127) / 128), 128, 0, st>>>(reinterpret_cast<const __half *>(w),
                                                                  reinterpret_cast<const __half *>(b), N, K, z,
                                                                  bfold);
    return cudaGetLastError();
}

cudaError_t launch_quantize_weights(const void *w, int64_t N, int64_t K, int bits_w, int8_t *qw, float *sw,
                                    cudaStream_t st) {
    if (N == 0) return cudaSuccess;
    const int iqmax = (1 << (bits_w - 1)) - 1;
    const int64_t grid = N < 65535 * 4 ? N : 65535 * 4;
    fold_codes_kernel<<<(unsigned)grid, kFoldThreads, 0, st>>>(reinterpret_cast<const __half *>(w), N, K, nullptr,
                                                               (float)iqmax, iqmax, qw, sw);
    return cudaGetLastError();
}

}  // namespace ot
