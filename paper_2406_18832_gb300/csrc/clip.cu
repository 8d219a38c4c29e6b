// clip.cu -- token-wise clipping calibration (Appendix D: the static
// activation scales of bias-free models are calibrated with token-wise
// clipping).  Per channel k of X_cal [T, K], with T' its non-NaN values and
// rho = ceil(alpha T') (fp64), the clipped range is [value of ascending rank
// T' + 1 - rho, value of ascending rank rho]: exact order statistics, so the
// result does not depend on how the work is split.
//
// Radix select on the 16-bit order-preserving key of each fp16 value (its bit
// pattern with the sign bit set for positives, all bits flipped for
// negatives): pass 1 histograms the key's top byte per channel, one thread
// per channel finds the bins holding both target ranks, pass 2 histograms the
// low byte inside those two bins and the ranks' exact keys follow.  A CTA owns
// a strip of 32 channels (lane = channel) and streams all T tokens of it
// twice; every histogram lives in shared memory (padded rows: lanes that hit
// the same bin use different banks), so no global scratch is needed.
#include <cuda_fp16.h>

#include <mutex>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

namespace {

constexpr int kClipThreads = 512;                 // 16 warps
constexpr int kClipWarps = kClipThreads / 32;
constexpr int kClipRows = 16;                     // token rows a warp loads before counting
constexpr int kClipPitch = 257;                   // padded histogram row

struct ClipSmem {
    unsigned coarse[32][kClipPitch];
    unsigned fine_lo[32][kClipPitch];
    unsigned fine_hi[32][kClipPitch];
    int bin_lo[32], bin_hi[32];
    long long rank_lo[32], rank_hi[32];           // ranks left inside the bins (1-based)
    int empty[32];
};

__device__ __forceinline__ bool is_nan_bits(unsigned short h) { return (h & 0x7C00u) == 0x7C00u && (h & 0x03FFu); }

__device__ __forceinline__ unsigned order_key(unsigned short h) {
    return (h & 0x8000u) ? (unsigned)(unsigned short)~h : (unsigned)(h | 0x8000u);
}

__device__ __forceinline__ unsigned short key_bits(unsigned key) {
    return (key & 0x8000u) ? (unsigned short)(key & 0x7FFFu) : (unsigned short)~key;
}

// Stream the strip's tokens: each warp takes kClipRows rows at a time (loads
// first, then counting).  pass 1: every key into coarse; pass 2: keys in the
// selected bins into the fine histograms.
template <bool kPass2>
__device__ __forceinline__ void clip_stream(const unsigned short *__restrict__ x, int64_t T, int64_t ldx, int64_t c,
                                           bool active, ClipSmem &S, int lane, int warp) {
    const int blo = kPass2 ? S.bin_lo[lane] : 0, bhi = kPass2 ? S.bin_hi[lane] : 0;
    for (int64_t t0 = (int64_t)warp * kClipRows; t0 < T; t0 += (int64_t)kClipWarps * kClipRows) {
        unsigned short v[kClipRows];
#pragma unroll
        for (int i = 0; i < kClipRows; ++i) {
            const int64_t t = t0 + i;
            v[i] = (active && t < T) ? __ldcs(x + t * ldx + c) : (unsigned short)0x7E00u;  // NaN: skipped
        }
#pragma unroll
        for (int i = 0; i < kClipRows; ++i) {
            if (is_nan_bits(v[i])) continue;
            const unsigned key = order_key(v[i]);
            const int top = (int)(key >> 8);
            if (!kPass2) {
                atomicAdd(&S.coarse[lane][top], 1u);
            } else {
                if (top == blo) atomicAdd(&S.fine_lo[lane][key & 255u], 1u);
                if (top == bhi) atomicAdd(&S.fine_hi[lane][key & 255u], 1u);
            }
        }
    }
}

__global__ void __launch_bounds__(kClipThreads) calibrate_clipped_kernel(const unsigned short *__restrict__ x,
                                                                         int64_t T, int64_t K, int64_t ldx,
                                                                         double alpha, float *lo, float *hi) {
    extern __shared__ unsigned char clip_smem_raw[];
    ClipSmem &S = *reinterpret_cast<ClipSmem *>(clip_smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t c = (int64_t)blockIdx.x * 32 + lane;
    const bool active = c < K;
    for (int i = threadIdx.x; i < 3 * 32 * kClipPitch; i += kClipThreads) (&S.coarse[0][0])[i] = 0u;
    __syncthreads();

    clip_stream<false>(x, T, ldx, c, active, S, lane, warp);
    __syncthreads();
    if (threadIdx.x < 32) {
        long long n = 0;
        for (int b = 0; b < 256; ++b) n += S.coarse[lane][b];
        S.empty[lane] = n == 0;
        long long rho = (long long)ceil(alpha * (double)n);
        rho = rho < 1 ? 1 : (rho > n ? n : rho);
        const long long r_hi = rho, r_lo = n + 1 - rho;
        long long cum = 0;
        int b_lo = 255, b_hi = 255;
        long long in_lo = 1, in_hi = 1;
        bool got_lo = false, got_hi = false;
        for (int b = 0; b < 256; ++b) {
            const long long next = cum + S.coarse[lane][b];
            if (!got_lo && next >= r_lo) {
                b_lo = b;
                in_lo = r_lo - cum;
                got_lo = true;
            }
            if (!got_hi && next >= r_hi) {
                b_hi = b;
                in_hi = r_hi - cum;
                got_hi = true;
            }
            cum = next;
        }
        S.bin_lo[lane] = b_lo;
        S.bin_hi[lane] = b_hi;
        S.rank_lo[lane] = in_lo;
        S.rank_hi[lane] = in_hi;
    }
    __syncthreads();

    clip_stream<true>(x, T, ldx, c, active, S, lane, warp);
    __syncthreads();
    if (threadIdx.x < 32 && active) {
        if (S.empty[lane]) {
            lo[c] = __int_as_float(0x7f800000);   // +inf
            hi[c] = __int_as_float(0xff800000);   // -inf
        } else {
            long long cum = 0;
            int low_lo = 255, low_hi = 255;
            bool got_lo = false, got_hi = false;
            for (int b = 0; b < 256; ++b) {
                const long long nlo = cum + S.fine_lo[lane][b];
                if (!got_lo && nlo >= S.rank_lo[lane]) {
                    low_lo = b;
                    got_lo = true;
                }
                cum = nlo;
            }
            cum = 0;
            for (int b = 0; b < 256; ++b) {
                const long long nhi = cum + S.fine_hi[lane][b];
                if (!got_hi && nhi >= S.rank_hi[lane]) {
                    low_hi = b;
                    got_hi = true;
                }
                cum = nhi;
            }
            const unsigned klo = ((unsigned)S.bin_lo[lane] << 8) | (unsigned)low_lo;
            const unsigned khi = ((unsigned)S.bin_hi[lane] << 8) | (unsigned)low_hi;
            lo[c] = __half2float(__ushort_as_half(key_bits(klo)));
            hi[c] = __half2float(__ushort_as_half(key_bits(khi)));
        }
    }
}

}  // namespace

cudaError_t launch_calibrate_clipped(const void *x, int64_t T, int64_t K, int64_t ldx, double alpha, float *lo,
                                     float *hi, cudaStream_t st) {
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [] {
        attr_err = cudaFuncSetAttribute(calibrate_clipped_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)sizeof(ClipSmem));
    });
    if (attr_err != cudaSuccess) return attr_err;
    const unsigned grid = (unsigned)((K + 31) / 32);
    calibrate_clipped_kernel<<<grid, kClipThreads, sizeof(ClipSmem), st>>>(
        reinterpret_cast<const unsigned short *>(x), T, K, ldx, alpha, lo, hi);
    return cudaGetLastError();
}

}  // namespace ot
