// calib.cu -- calibration (per-channel min / max, Appendix A) and the static
// per-channel parameters z, s, r (Section 3.2; Eq. 1 with zero point 0).
#include <cuda_fp16.h>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

namespace {

// Float min / max through integer atomics.  For a float with the sign bit
// clear, signed-int order equals float order and every float with the sign
// bit set compares below it as a signed int; for sign-bit-set floats,
// unsigned order is the reverse of float order.  NaN never reaches these.
__device__ __forceinline__ void atomic_min_f32(float *addr, float v) {
    if (!(__float_as_uint(v) >> 31))
        atomicMin(reinterpret_cast<int *>(addr), __float_as_int(v));
    else
        atomicMax(reinterpret_cast<unsigned *>(addr), __float_as_uint(v));
}
__device__ __forceinline__ void atomic_max_f32(float *addr, float v) {
    if (!(__float_as_uint(v) >> 31))
        atomicMax(reinterpret_cast<int *>(addr), __float_as_int(v));
    else
        atomicMin(reinterpret_cast<unsigned *>(addr), __float_as_uint(v));
}

__global__ void reset_minmax_kernel(float *mn, float *mx, int64_t K) {
    int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (k < K) {
        mn[k] = __int_as_float(0x7f800000);   // +inf
        mx[k] = __int_as_float(0xff800000);   // -inf
    }
}

// Block: 32 x 8 threads.  threadIdx.x owns 8 consecutive channels (one 16-byte
// vector); a warp spans 256 channels (512 contiguous bytes of a row) and the
// 8 warps stride over rows.  blockIdx.x picks the 256-channel strip,
// blockIdx.y a contiguous range of rows.  fp16 min / max are exact, and
// __hmin2 / __hmax2 return the non-NaN operand, so NaN is ignored.
constexpr int kCalRowsUnroll = 4;

__global__ void __launch_bounds__(256) calibrate_kernel(const __half *__restrict__ x, int64_t T, int64_t K,
                                                        int64_t ldx, int64_t rows_per_block, float *mn,
                                                        float *mx) {
    __shared__ float s_mn[8][256];
    __shared__ float s_mx[8][256];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int64_t c0 = (int64_t)blockIdx.x * 256 + tx * 8;
    const int64_t r_begin = (int64_t)blockIdx.y * rows_per_block;
    const int64_t r_end = min(T, r_begin + rows_per_block);
    const __half2 pinf = __halves2half2(__ushort_as_half(0x7c00), __ushort_as_half(0x7c00));
    const __half2 ninf = __halves2half2(__ushort_as_half(0xfc00), __ushort_as_half(0xfc00));
    __half2 lo[4] = {pinf, pinf, pinf, pinf}, hi[4] = {ninf, ninf, ninf, ninf};
    if (c0 < K) {
        const __half *base = x + c0;
        int64_t r = r_begin + ty;
        for (; r + 8 * (kCalRowsUnroll - 1) < r_end; r += 8 * kCalRowsUnroll) {
            uint4 v[kCalRowsUnroll];
#pragma unroll
            for (int u = 0; u < kCalRowsUnroll; ++u)
                v[u] = __ldcs(reinterpret_cast<const uint4 *>(base + (r + 8 * u) * ldx));
#pragma unroll
            for (int u = 0; u < kCalRowsUnroll; ++u) {
                const __half2 *h = reinterpret_cast<const __half2 *>(&v[u]);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    lo[j] = __hmin2(lo[j], h[j]);
                    hi[j] = __hmax2(hi[j], h[j]);
                }
            }
        }
        for (; r < r_end; r += 8) {
            uint4 v = __ldcs(reinterpret_cast<const uint4 *>(base + r * ldx));
            const __half2 *h = reinterpret_cast<const __half2 *>(&v);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                lo[j] = __hmin2(lo[j], h[j]);
                hi[j] = __hmax2(hi[j], h[j]);
            }
        }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        s_mn[ty][tx * 8 + 2 * j] = __low2float(lo[j]);
        s_mn[ty][tx * 8 + 2 * j + 1] = __high2float(lo[j]);
        s_mx[ty][tx * 8 + 2 * j] = __low2float(hi[j]);
        s_mx[ty][tx * 8 + 2 * j + 1] = __high2float(hi[j]);
    }
    __syncthreads();
    const int c = threadIdx.x;  // 256 threads, one channel of the strip each
    const int64_t k = (int64_t)blockIdx.x * 256 + c;
    if (k < K) {
        float a = s_mn[0][c], b = s_mx[0][c];
#pragma unroll
        for (int w = 1; w < 8; ++w) {
            a = fminf(a, s_mn[w][c]);
            b = fmaxf(b, s_mx[w][c]);
        }
        if (a != __int_as_float(0x7f800000)) atomic_min_f32(mn + k, a);
        if (b != __int_as_float(0xff800000)) atomic_max_f32(mx + k, b);
    }
}

__global__ void params_kernel(const float *__restrict__ mn, const float *__restrict__ mx, int64_t K, float qmax,
                              int symmetrize, float *z, float *s, float *r) {
    int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (k >= K) return;
    const float lo = mn[k], hi = mx[k];
    if (!(lo <= hi) || isinf(lo) || isinf(hi)) {
        z[k] = 0.f;
        s[k] = 0.f;
        r[k] = 0.f;
        return;
    }
    float zk, amp;
    if (symmetrize) {
        zk = __fmul_rn(__fadd_rn(hi, lo), 0.5f);
        amp = fmaxf(__fsub_rn(hi, zk), __fsub_rn(zk, lo));
    } else {
        zk = 0.f;
        amp = fmaxf(fabsf(hi), fabsf(lo));
    }
    z[k] = zk;
    if (amp > 0.f && isfinite(amp)) {
        s[k] = __fdiv_rn(amp, qmax);
        r[k] = __fdiv_rn(qmax, amp);
    } else {
        s[k] = 0.f;
        r[k] = 0.f;
    }
}

}  // namespace

cudaError_t launch_calibrate(const void *x, int64_t T, int64_t K, int64_t ldx, float *mn, float *mx, int reset,
                             cudaStream_t st) {
    if (reset) {
        reset_minmax_kernel<<<(unsigned)((K + 255) / 256), 256, 0, st>>>(mn, mx, K);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (T == 0) return cudaSuccess;
    const int64_t strips = (K + 255) / 256;
    // enough CTAs for every SM to hold several, each with a long run of rows
    int64_t want = (int64_t)num_sms() * 8;
    int64_t splits = (want + strips - 1) / strips;
    int64_t max_splits = (T + 63) / 64;  // at least 64 rows per CTA
    if (splits > max_splits) splits = max_splits;
    if (splits < 1) splits = 1;
    if (splits > 65535) splits = 65535;
    const int64_t rows = (T + splits - 1) / splits;
    splits = (T + rows - 1) / rows;
    dim3 grid((unsigned)strips, (unsigned)splits);
    calibrate_kernel<<<grid, 256, 0, st>>>(reinterpret_cast<const __half *>(x), T, K, ldx, rows, mn, mx);
    return cudaGetLastError();
}

cudaError_t launch_params(const float *mn, const float *mx, int64_t K, int bits, int symmetrize, float *z,
                          float *s, float *r, cudaStream_t st) {
    const float qmax = (float)((1 << (bits - 1)) - 1);
    params_kernel<<<(unsigned)((K + 255) / 256), 256, 0, st>>>(mn, mx, K, qmax, symmetrize, z, s, r);
    return cudaGetLastError();
}

}  // namespace ot
