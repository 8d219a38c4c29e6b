// layernorm.cu -- the LayerNorm before a per-channel quantized linear, fused
// with the symmetrization and the activation quantization (Section 3.2: the
// codes round(X_hat / s) "through the kernel fusion with its previous
// LayerNorm"; LN's gamma and beta absorb r and z):
//   q = round(((h - mean) * rstd) * gamma_r + beta_r),
//   gamma_r = gamma * r,  beta_r = (beta - z) * r   (folded once, offline).
// The row statistics are exact so the codes do not depend on a reduction
// order: h * 2^24 is an integer H for every fp16 h (|H| < 2^40), split as
// H = A 2^20 + B with |A| <= 2^20, |B| <= 2^19 (h rounded to a multiple of
// 2^-4, and the rest); sum H is kept as the exact sums of A and of B, and
// sum H^2 = 2^40 sum A^2 + 2^21 sum AB + sum B^2 as three exact 64-bit sums,
// combined in 128 bits once per row.  Mean and 1/sqrt(var + eps) then follow
// by a fixed sequence of IEEE fp32 operations (one lane per row) and the
// codes by one fp32 fma per element.
// Rows up to 16384 wide are held in registers by one to eight warps (one HBM
// read with the whole row in flight), longer ones are streamed by one warp
// and read again from L2 for the codes.
#include <cuda_fp16.h>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

namespace {

constexpr int kLnThreads = 256;
constexpr int kLnWarps = kLnThreads / 32;  // rows per CTA

__global__ void __launch_bounds__(256) fold_layernorm_kernel(const __half *__restrict__ gamma,
                                                             const __half *__restrict__ beta,
                                                             const float *__restrict__ z,
                                                             const float *__restrict__ r, int64_t K,
                                                             float *gamma_r, float *beta_r) {
    const int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (k >= K) return;
    const float rk = __ldg(r + k);
    gamma_r[k] = __fmul_rn(__half2float(gamma[k]), rk);
    beta_r[k] = __fmul_rn(__fsub_rn(__half2float(beta[k]), __ldg(z + k)), rk);
}

struct LnSums {
    long long s1;                 // S1 = sum H = 2^20 sum A + sum B
    unsigned long long a, b, c;   // sum A^2, sum AB (two's complement), sum B^2
    int bad;                      // non-finite values seen
};

// The split of fp16 values h (exact in fp32) into A and B, all in fp32 adds
// whose results are exact (the splitting of Rump, Ogita and Oishi,
// "Accurate floating-point summation", SIAM J. Sci. Comput. 31 (2008)):
// t1 = h + 1.5 2^19 lies in [2^19, 2^20), where fp32 values are 2^-4 apart,
// so t1 - 1.5 2^19 = h_hi is h rounded to a multiple of 2^-4 and h_lo =
// h - h_hi (|h_lo| <= 2^-5, a multiple of 2^-24) is exact; t2 = h_lo + 0.75
// lies in [0.5, 1), where values are 2^-24 apart, and is exact too.  Within
// one binade the bit pattern grows by one per spacing, so A = bits(t1) -
// bits(1.5 2^19) = 16 h_hi and B = bits(t2) - bits(0.75) = 2^24 h_lo.  An
// infinite or NaN h makes h_lo and t2 NaN, whose pattern has bit 30 set;
// every finite t2 has it clear.  Two values per fp32x2 instruction.
constexpr uint32_t kLnBitsHi = 0x49400000u;  // 1.5 * 2^19
constexpr uint32_t kLnBitsLo = 0x3F400000u;  // 0.75

__device__ __forceinline__ void ln_take(uint32_t u1, uint32_t u2, uint32_t &sa, uint32_t &sb, uint32_t &nf,
                                        LnSums &s) {
    sa += u1;  // wrapping: the chunk's true sum fits in 32 bits
    sb += u2;
    nf |= u2;
    const int A = (int)(u1 - kLnBitsHi), B = (int)(u2 - kLnBitsLo);
    s.a += (unsigned long long)((long long)A * A);
    s.b += (unsigned long long)((long long)A * B);
    s.c += (unsigned long long)((long long)B * B);
}

// One 16-byte chunk (8 values) into the sums; |sum A| <= 2^23 and
// |sum B| <= 2^22 over the chunk, so the sums of the bit patterns, minus 8
// times the addends' patterns, are exact modulo 2^32 and in range.
__device__ __forceinline__ void ln_add8(LnSums &s, const uint4 &d) {
    uint32_t sa = 0, sb = 0, nf = 0;
    const __half2 *hv = reinterpret_cast<const __half2 *>(&d);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 x = __half22float2(hv[j]);
        const float2 t1 = f2_add(x, make_float2(786432.0f, 786432.0f));
        const float2 hi = f2_add(t1, make_float2(-786432.0f, -786432.0f));
        const float2 t2 = f2_add(f2_fma(hi, make_float2(-1.0f, -1.0f), x), make_float2(0.75f, 0.75f));
        ln_take(__float_as_uint(t1.x), __float_as_uint(t2.x), sa, sb, nf, s);
        ln_take(__float_as_uint(t1.y), __float_as_uint(t2.y), sa, sb, nf, s);
    }
    s.s1 += (long long)(int)(sa - 8u * kLnBitsHi) * (1LL << 20) + (int)(sb - 8u * kLnBitsLo);
    s.bad |= (int)((nf >> 30) & 1u);
}

// Codes of 8 elements (one 16-byte chunk of the row) from mean, rstd and the
// folded affine; returns their sum.  Per element, as in the scalar form:
// n = fl(fl(h - mean) * rstd), u = fma(n, gamma_r, beta_r), two per fp32x2
// instruction.
template <bool kF16Out>
__device__ __forceinline__ int ln_codes8(const uint4 &d, int64_t k, float mean, float rstd,
                                         const float *__restrict__ gamma_r, const float *__restrict__ beta_r,
                                         int qmax, void *q, int64_t qoff, bool bad) {
    int c[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    if (!bad) {
        const __half2 *hv = reinterpret_cast<const __half2 *>(&d);
        const float4 g0 = __ldg(reinterpret_cast<const float4 *>(gamma_r + k));
        const float4 g1 = __ldg(reinterpret_cast<const float4 *>(gamma_r + k + 4));
        const float4 b0 = __ldg(reinterpret_cast<const float4 *>(beta_r + k));
        const float4 b1 = __ldg(reinterpret_cast<const float4 *>(beta_r + k + 4));
        const float2 g[4] = {make_float2(g0.x, g0.y), make_float2(g0.z, g0.w), make_float2(g1.x, g1.y),
                             make_float2(g1.z, g1.w)};
        const float2 bb[4] = {make_float2(b0.x, b0.y), make_float2(b0.z, b0.w), make_float2(b1.x, b1.y),
                              make_float2(b1.z, b1.w)};
        const float2 nm = make_float2(-mean, -mean), rs2 = make_float2(rstd, rstd);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 n = f2_mul(f2_add(__half22float2(hv[j]), nm), rs2);
            const float2 u = f2_fma(n, g[j], bb[j]);
            // cvt.rni maps NaN to 0 and saturates; then the symmetric range
            c[2 * j] = max(-qmax, min(qmax, __float2int_rn(u.x)));
            c[2 * j + 1] = max(-qmax, min(qmax, __float2int_rn(u.y)));
        }
    }
    int rs = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) rs += c[j];
    if (kF16Out) {
        // fp16 holding the integer c: the pattern 0x6400 | (c + 128), minus 1152 (exact)
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t bits = (uint32_t)(0x6480 + c[2 * j]) | ((uint32_t)(0x6480 + c[2 * j + 1]) << 16);
            const __half2 v = __hsub2(*reinterpret_cast<const __half2 *>(&bits),
                                      __half2half2(__ushort_as_half(0x6480)));
            w[j] = *reinterpret_cast<const uint32_t *>(&v);
        }
        *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(q) + qoff) = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
        uint2 o;
        o.x = __byte_perm(__byte_perm((uint32_t)c[0], (uint32_t)c[1], 0x0040),
                          __byte_perm((uint32_t)c[2], (uint32_t)c[3], 0x0040), 0x5410);
        o.y = __byte_perm(__byte_perm((uint32_t)c[4], (uint32_t)c[5], 0x0040),
                          __byte_perm((uint32_t)c[6], (uint32_t)c[7], 0x0040), 0x5410);
        *reinterpret_cast<uint2 *>(reinterpret_cast<int8_t *>(q) + qoff) = o;
    }
    return rs;
}

// The warp's sums, added over its lanes (exact).
__device__ __forceinline__ void ln_warp_reduce(LnSums &s) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        s.s1 += __shfl_xor_sync(0xffffffffu, s.s1, o);
        s.a += __shfl_xor_sync(0xffffffffu, s.a, o);
        s.b += __shfl_xor_sync(0xffffffffu, s.b, o);
        s.c += __shfl_xor_sync(0xffffffffu, s.c, o);
    }
    s.bad = __any_sync(0xffffffffu, s.bad);
}

// mean and rstd of a row from its exact sums, by IEEE fp32 operations in
// the order documented above (one thread).
__device__ __forceinline__ void ln_moments(const LnSums &s, int64_t K, float eps, float &mean, float &rstd) {
    const float kf = (float)K;  // exact: K <= 2^22
    mean = __fmul_rn(__fdiv_rn(__ll2float_rn(s.s1), kf), 0x1p-24f);  // exact S1: |S1| < 2^62
    const __int128 s2 = ((__int128)s.a << 40) + ((__int128)(long long)s.b << 21) + (__int128)s.c;
    const __int128 s1 = (__int128)s.s1;
    const unsigned __int128 v = (unsigned __int128)((__int128)K * s2 - s1 * s1);  // >= 0 (Cauchy-Schwarz)
    const float vf = __fadd_rn(__fmul_rn(__ull2float_rn((unsigned long long)(v >> 64)), 18446744073709551616.0f),
                               __ull2float_rn((unsigned long long)v));
    const float var = __fmul_rn(__fdiv_rn(__fdiv_rn(vf, kf), kf), 0x1p-48f);
    rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, eps)));
}

// The warp's sums reduced, the moments taken by lane 0 and broadcast.
__device__ __forceinline__ void ln_stats(LnSums &s, int64_t K, float eps, float &mean, float &rstd) {
    ln_warp_reduce(s);
    mean = 0.f;
    rstd = 0.f;
    if ((threadIdx.x & 31) == 0 && !s.bad) ln_moments(s, K, eps, mean, rstd);
    mean = __shfl_sync(0xffffffffu, mean, 0);
    rstd = __shfl_sync(0xffffffffu, rstd, 0);
}

// kWpr warps per row (kLnWarps / kWpr rows per CTA, grid-stride): lane l of
// the row's warp w holds the 16-byte chunks l + 32 (i kWpr + w), i < kCh, in
// registers (K <= 256 kWpr kCh).  Each warp adds its share of the exact sums;
// the shares meet in shared memory, the row's first warp alone adds them and
// takes the moments (a serial chain of 128-bit integer and fp32 division
// steps, which the other warps would only repeat), and its result reaches
// the row's warps through shared memory: two named barriers per row.  The
// sums are exact, so the result is that of one warp over the whole row.
// Four 256-thread CTAs per SM (64 registers) for every width up to 8192,
// with four chunks per lane (measured on GB300: 2048 x 7168 in 21.9 us with
// eight warps per row against 23.7 us with four warps of eight chunks); two
// CTAs per SM with six or eight chunks per lane of eight warps up to 16384
// (against the streaming kernel below: 4096 x 9216 62 vs 69 us, 2048 x 12288
// 38 vs 41 us, 2048 x 16384 48 vs 58 us; 2048 x 9216 32 vs 31 us).
template <bool kF16Out, int kCh, int kWpr>
__global__ void __launch_bounds__(kLnThreads, kCh <= 4 ? 4 : 2) layernorm_quantize_rows_kernel(
    const __half *__restrict__ h, int64_t M, int64_t K, int64_t ldh, const float *__restrict__ gamma_r,
    const float *__restrict__ beta_r, float eps, int qmax, void *q, int32_t *rowsum) {
    // launched as a programmatic dependent: the kernel before this one has
    // written h; the next one starts only after that (see quantize_kernel)
    grid_dep_wait();
    grid_dep_launch();
    constexpr int kRows = kLnWarps / kWpr;
    __shared__ LnSums part[kLnWarps];
    __shared__ float2 stat[kRows];  // mean, rstd; rstd is NaN for a row with non-finite values
    __shared__ int rsum[kLnWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rr = warp / kWpr, w = warp % kWpr;  // row of the CTA, warp of the row
    const int bar = 1 + rr;                        // named barrier of the row's warps
    for (int64_t m = (int64_t)blockIdx.x * kRows + rr; m < M; m += (int64_t)gridDim.x * kRows) {
        const __half *row = h + m * ldh;
        LnSums s{0, 0, 0, 0, 0};
        uint4 d[kCh];
#pragma unroll
        for (int i = 0; i < kCh; ++i) {
            const int64_t k = (int64_t)(lane + 32 * (i * kWpr + w)) * 8;
            d[i] = k < K ? __ldcs(reinterpret_cast<const uint4 *>(row + k)) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int i = 0; i < kCh; ++i)
            if ((int64_t)(lane + 32 * (i * kWpr + w)) * 8 < K) ln_add8(s, d[i]);
        float mean, rstd;
        bool bad;
        if (kWpr > 1) {
            ln_warp_reduce(s);
            if (lane == 0) part[warp] = s;
            asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(32 * kWpr) : "memory");
            if (w == 0 && lane == 0) {
                LnSums t = part[rr * kWpr];
#pragma unroll
                for (int v = 1; v < kWpr; ++v) {
                    const LnSums &o = part[rr * kWpr + v];
                    t.s1 += o.s1;
                    t.a += o.a;
                    t.b += o.b;
                    t.c += o.c;
                    t.bad |= o.bad;
                }
                float mu = 0.f, rs = __int_as_float(0x7fffffff);
                if (!t.bad) ln_moments(t, K, eps, mu, rs);
                stat[rr] = make_float2(mu, rs);
            }
            asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(32 * kWpr) : "memory");
            const float2 st = stat[rr];
            mean = st.x;
            rstd = st.y;
            bad = rstd != rstd;
        } else {
            ln_stats(s, K, eps, mean, rstd);
            bad = s.bad != 0;
        }
        int rs = 0;
#pragma unroll
        for (int i = 0; i < kCh; ++i) {
            const int64_t k = (int64_t)(lane + 32 * (i * kWpr + w)) * 8;
            if (k < K) rs += ln_codes8<kF16Out>(d[i], k, mean, rstd, gamma_r, beta_r, qmax, q, m * K + k, bad);
        }
        if (rowsum) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) rs += __shfl_xor_sync(0xffffffffu, rs, o);
            if (kWpr > 1) {
                if (lane == 0) rsum[warp] = rs;
                asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(32 * kWpr) : "memory");
                if (w == 0 && lane == 0) {
                    int t = 0;
#pragma unroll
                    for (int v = 0; v < kWpr; ++v) t += rsum[rr * kWpr + v];
                    rowsum[m] = t;
                }
            } else if (lane == 0) {
                rowsum[m] = rs;
            }
        }
        // the shares of this row may be overwritten by the next row only after every warp read them
        if (kWpr > 1) asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(32 * kWpr) : "memory");
    }
}

// One warp per row (kLnWarps rows per CTA, grid-stride).  kCh > 0: the lane
// holds its kCh 16-byte chunks of the row (K <= 256 kCh) in registers, all
// loaded before use, so the row is read from HBM once with the whole row in
// flight.  kCh == 0: longer rows stream in batches of 8 chunks per lane and
// are read again (from L2) for the codes.
template <bool kF16Out, int kCh>
__global__ void __launch_bounds__(kLnThreads) layernorm_quantize_kernel(const __half *__restrict__ h, int64_t M,
                                                                        int64_t K, int64_t ldh,
                                                                        const float *__restrict__ gamma_r,
                                                                        const float *__restrict__ beta_r, float eps,
                                                                        int qmax, void *q, int32_t *rowsum) {
    grid_dep_wait();
    grid_dep_launch();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int64_t m = (int64_t)blockIdx.x * kLnWarps + warp; m < M; m += (int64_t)gridDim.x * kLnWarps) {
        const __half *row = h + m * ldh;
        LnSums s{0, 0, 0, 0, 0};
        float mean, rstd;
        int rs = 0;
        if constexpr (kCh > 0) {
            uint4 d[kCh];
#pragma unroll
            for (int i = 0; i < kCh; ++i) {
                const int64_t k = (int64_t)(lane + 32 * i) * 8;
                d[i] = k < K ? __ldcs(reinterpret_cast<const uint4 *>(row + k)) : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
            for (int i = 0; i < kCh; ++i)
                if ((int64_t)(lane + 32 * i) * 8 < K) ln_add8(s, d[i]);
            ln_stats(s, K, eps, mean, rstd);
#pragma unroll
            for (int i = 0; i < kCh; ++i) {
                const int64_t k = (int64_t)(lane + 32 * i) * 8;
                if (k < K) rs += ln_codes8<kF16Out>(d[i], k, mean, rstd, gamma_r, beta_r, qmax, q, m * K + k, s.bad);
            }
        } else {
            constexpr int kB = 8;
            for (int64_t k0 = (int64_t)lane * 8; k0 < K; k0 += 32 * 8 * kB) {
                uint4 d[kB];
#pragma unroll
                for (int i = 0; i < kB; ++i) {
                    const int64_t k = k0 + (int64_t)i * 32 * 8;
                    d[i] = k < K ? __ldg(reinterpret_cast<const uint4 *>(row + k)) : make_uint4(0, 0, 0, 0);
                }
#pragma unroll
                for (int i = 0; i < kB; ++i)
                    if (k0 + (int64_t)i * 32 * 8 < K) ln_add8(s, d[i]);
            }
            ln_stats(s, K, eps, mean, rstd);
            for (int64_t k0 = (int64_t)lane * 8; k0 < K; k0 += 32 * 8 * kB) {
                uint4 d[kB];
#pragma unroll
                for (int i = 0; i < kB; ++i) {
                    const int64_t k = k0 + (int64_t)i * 32 * 8;
                    d[i] = k < K ? __ldcs(reinterpret_cast<const uint4 *>(row + k)) : make_uint4(0, 0, 0, 0);
                }
#pragma unroll
                for (int i = 0; i < kB; ++i) {
                    const int64_t k = k0 + (int64_t)i * 32 * 8;
                    if (k < K) rs += ln_codes8<kF16Out>(d[i], k, mean, rstd, gamma_r, beta_r, qmax, q, m * K + k, s.bad);
                }
            }
        }
        if (rowsum) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) rs += __shfl_xor_sync(0xffffffffu, rs, o);
            if (lane == 0) rowsum[m] = rs;
        }
    }
}

template <bool kF16Out>
cudaError_t run_layernorm_quantize(const __half *h, int64_t M, int64_t K, int64_t ldh, const float *gamma_r,
                                   const float *beta_r, float eps, int qmax, void *q, int32_t *rowsum,
                                   cudaStream_t st) {
    const int64_t ch = (K + 255) / 256;  // 16-byte chunks per lane of one warp
    auto grid_for = [&](int rows_per_cta) {
        const int64_t ctas = (M + rows_per_cta - 1) / rows_per_cta;
        return (unsigned)(ctas < (1 << 30) ? ctas : (1 << 30));
    };
#define OT_LN_ROWS(C, W)                                                                                      \
    launch_kernel(layernorm_quantize_rows_kernel<kF16Out, C, W>, dim3(grid_for(kLnWarps / W)), dim3(kLnThreads), 0, \
                  st, true, h, M, K, ldh, gamma_r, beta_r, eps, qmax, q, rowsum)
    if (ch <= 4) return OT_LN_ROWS(4, 1);
    if (ch <= 8) return OT_LN_ROWS(4, 2);
    if (ch <= 16) return OT_LN_ROWS(4, 4);
    if (ch <= 32) return OT_LN_ROWS(4, 8);
    if (ch <= 48) return OT_LN_ROWS(6, 8);
    if (ch <= 64) return OT_LN_ROWS(8, 8);
#undef OT_LN_ROWS
    return launch_kernel(layernorm_quantize_kernel<kF16Out, 0>, dim3(grid_for(kLnWarps)), dim3(kLnThreads), 0, st, true,
                         h, M, K, ldh, gamma_r, beta_r, eps, qmax, q, rowsum);
}

}  // namespace

cudaError_t launch_fold_layernorm(const void *gamma, const void *beta, const float *z, const float *r, int64_t K,
                                  float *gamma_r, float *beta_r, cudaStream_t st) {
    fold_layernorm_kernel<<<(unsigned)((K + 255) / 256), 256, 0, st>>>(
        reinterpret_cast<const __half *>(gamma), reinterpret_cast<const __half *>(beta), z, r, K, gamma_r, beta_r);
    return cudaGetLastError();
}

cudaError_t launch_layernorm_quantize(const void *h, int64_t M, int64_t K, int64_t ldh, const float *gamma_r,
                                      const float *beta_r, float eps, int bits, void *q, int fmt,
                                      int32_t *rowsum, cudaStream_t st) {
    if (M == 0) return cudaSuccess;
    const int qmax = (1 << (bits - 1)) - 1;
    const __half *hh = reinterpret_cast<const __half *>(h);
    if (fmt == OT_CODE_F16) return run_layernorm_quantize<true>(hh, M, K, ldh, gamma_r, beta_r, eps, qmax, q, rowsum, st);
    return run_layernorm_quantize<false>(hh, M, K, ldh, gamma_r, beta_r, eps, qmax, q, rowsum, st);
}

}  // namespace ot
