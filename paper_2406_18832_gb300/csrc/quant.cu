// quant.cu -- per-channel static activation quantization, round(X_hat / s)
// with X_hat = X - z (Eq. 6, Eq. 7): q = clamp(rne((x - z_k) * r_k)).
// HBM-bound: one 16-byte fp16 load and one 16-byte (fp16 codes) or 8-byte
// (int8 codes) store per 8 elements, coalesced across the warp.
#include <cuda_fp16.h>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

OT_DEBUG_UNIT(quant)

namespace {

constexpr int kQRowsPerThread = 8;              // rows a thread walks with the same z, r
constexpr int kQRowsPerBlock = 8 * kQRowsPerThread;

__device__ __forceinline__ int code_of(float x, float z, float r, int qmax) {
    // two fp32 roundings as written (no contraction), then round half to even;
    // cvt.rni.s32.f32 maps NaN to 0 and saturates out-of-range values
    const float u = __fmul_rn(__fsub_rn(x, z), r);
    const int c = __float2int_rn(u);
    return max(-qmax, min(qmax, c));
}

// fp16 holding the integer c (|c| <= 128): 1152 + c lies in [1024, 2048) where
// fp16 has unit spacing, so its bit pattern is 0x6400 | (128 + c); subtracting
// 1152 in fp16 is exact.
__device__ __forceinline__ uint32_t pack_f16_codes(int c0, int c1) {
    const uint32_t bits = (uint32_t)(0x6480 + c0) | ((uint32_t)(0x6480 + c1) << 16);
    const __half2 v = __hsub2(*reinterpret_cast<const __half2 *>(&bits), __half2half2(__ushort_as_half(0x6480)));
    return *reinterpret_cast<const uint32_t *>(&v);
}

__device__ __forceinline__ uint32_t pack_i8_codes(int c0, int c1, int c2, int c3) {
    const uint32_t lo = __byte_perm((uint32_t)c0, (uint32_t)c1, 0x0040);
    const uint32_t hi = __byte_perm((uint32_t)c2, (uint32_t)c3, 0x0040);
    return __byte_perm(lo, hi, 0x5410);
}

// Block 32 x 8: threadIdx.x owns 8 consecutive channels of a 256-channel
// strip (blockIdx.x) and keeps their z, r in registers while it walks
// kQRowsPerThread rows of the block's row range (blockIdx.y).  With kRowSum
// the warp also adds its 256 codes of each row and one lane adds that into
// rowsum[m] (integer atomics: exact, order-free; rowsum starts at 0).
template <bool kF16Out, bool kRowSum>
__global__ void __launch_bounds__(256) quantize_kernel(const __half *__restrict__ x, int64_t M, int64_t K,
                                                       int64_t ldx, const float *__restrict__ z,
                                                       const float *__restrict__ r, int qmax, void *q,
                                                       int32_t *rowsum) {
    // Launched as a programmatic dependent: wait for the kernel before this one
    // (its writes of x, z, r), then let the next one start -- only then, so a
    // dependent linear that loads its weights before its own wait starts after
    // every earlier kernel (any writer of the weights) has completed.
    grid_dep_wait();
    grid_dep_launch();
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int64_t c0 = (int64_t)blockIdx.x * 256 + tx * 8;
    const bool active = c0 < K;  // K % 8 == 0: a lane's 8 channels are whole or absent
    if (!kRowSum && !active) return;
    float zz[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f}, rr[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (active) {
        const float4 *zp = reinterpret_cast<const float4 *>(z + c0);
        const float4 *rp = reinterpret_cast<const float4 *>(r + c0);
        float4 a = __ldg(zp), b = __ldg(zp + 1), c = __ldg(rp), d = __ldg(rp + 1);
        zz[0] = a.x; zz[1] = a.y; zz[2] = a.z; zz[3] = a.w; zz[4] = b.x; zz[5] = b.y; zz[6] = b.z; zz[7] = b.w;
        rr[0] = c.x; rr[1] = c.y; rr[2] = c.z; rr[3] = c.w; rr[4] = d.x; rr[5] = d.y; rr[6] = d.z; rr[7] = d.w;
    }
    const int64_t row0 = (int64_t)blockIdx.y * kQRowsPerBlock + ty;
    uint4 v[kQRowsPerThread];
#pragma unroll
    for (int u = 0; u < kQRowsPerThread; ++u) {
        const int64_t m = row0 + 8 * u;
        v[u] = make_uint4(0, 0, 0, 0);
        if (m < M && active) v[u] = __ldcs(reinterpret_cast<const uint4 *>(x + m * ldx + c0));
    }
#pragma unroll
    for (int u = 0; u < kQRowsPerThread; ++u) {
        const int64_t m = row0 + 8 * u;
        if (m >= M) break;  // uniform over the warp
        const __half2 *h = reinterpret_cast<const __half2 *>(&v[u]);
        int c[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 f = __half22float2(h[j]);
            c[2 * j] = code_of(f.x, zz[2 * j], rr[2 * j], qmax);
            c[2 * j + 1] = code_of(f.y, zz[2 * j + 1], rr[2 * j + 1], qmax);
        }
        if (kRowSum) {
            int t = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) t += c[j];  // inactive lanes: codes of 0 * 0 = 0
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            if (tx == 0) atomicAdd(rowsum + m, t);
        }
        if (!active) continue;
        if (kF16Out) {
            uint4 o;
            o.x = pack_f16_codes(c[0], c[1]);
            o.y = pack_f16_codes(c[2], c[3]);
            o.z = pack_f16_codes(c[4], c[5]);
            o.w = pack_f16_codes(c[6], c[7]);
            if (OT_DCHECK(m < M && c0 + 8 <= K))
                *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(q) + m * K + c0) = o;
        } else {
            uint2 o;
            o.x = pack_i8_codes(c[0], c[1], c[2], c[3]);
            o.y = pack_i8_codes(c[4], c[5], c[6], c[7]);
            if (OT_DCHECK(m < M && c0 + 8 <= K))
                *reinterpret_cast<uint2 *>(reinterpret_cast<int8_t *>(q) + m * K + c0) = o;
        }
    }
}

// Per-token dynamic quantization (Eq. 3; Eq. 1 with zero point 0 and one
// scale per row): one CTA per row; pass 1 takes amax = max |x| (fp16 max is
// exact; __hmax2 returns the non-NaN operand), pass 2 re-reads the row (L2 /
// L1 hit) and writes round(x * r) with r = qmax / amax.
template <bool kF16Out>
__global__ void __launch_bounds__(256) quantize_tokens_kernel(const __half *__restrict__ x, int64_t K, int64_t ldx,
                                                              int qmax, void *q, float *s_tok) {
    __shared__ float red[8];
    const int64_t m = blockIdx.x;
    const __half *row = x + m * ldx;
    const int64_t nv = K / 8;
    __half2 hm = __float2half2_rn(0.f);
    for (int64_t v = threadIdx.x; v < nv; v += 256) {
        const uint4 d = __ldg(reinterpret_cast<const uint4 *>(row + v * 8));
        const __half2 *h = reinterpret_cast<const __half2 *>(&d);
#pragma unroll
        for (int j = 0; j < 4; ++j) hm = __hmax2(hm, __habs2(h[j]));
    }
    float a = fmaxf(__low2float(hm), __high2float(hm));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = a;
    __syncthreads();
    float amax = red[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) amax = fmaxf(amax, red[w]);
    float s = 0.f, r = 0.f;
    if (amax > 0.f && isfinite(amax)) {
        s = __fdiv_rn(amax, (float)qmax);
        r = __fdiv_rn((float)qmax, amax);
    }
    if (threadIdx.x == 0) s_tok[m] = s;
    for (int64_t v = threadIdx.x; v < nv; v += 256) {
        const uint4 d = __ldg(reinterpret_cast<const uint4 *>(row + v * 8));
        const __half2 *h = reinterpret_cast<const __half2 *>(&d);
        int c[8];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float2 f = __half22float2(h[j]);
            c[2 * j] = max(-qmax, min(qmax, __float2int_rn(__fmul_rn(f.x, r))));
            c[2 * j + 1] = max(-qmax, min(qmax, __float2int_rn(__fmul_rn(f.y, r))));
        }
        if (kF16Out) {
            uint4 o;
            o.x = pack_f16_codes(c[0], c[1]);
            o.y = pack_f16_codes(c[2], c[3]);
            o.z = pack_f16_codes(c[4], c[5]);
            o.w = pack_f16_codes(c[6], c[7]);
            if (OT_DCHECK(v * 8 + 8 <= K))
                *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(q) + m * K + v * 8) = o;
        } else {
            uint2 o;
            o.x = pack_i8_codes(c[0], c[1], c[2], c[3]);
            o.y = pack_i8_codes(c[4], c[5], c[6], c[7]);
            if (OT_DCHECK(v * 8 + 8 <= K))
                *reinterpret_cast<uint2 *>(reinterpret_cast<int8_t *>(q) + m * K + v * 8) = o;
        }
    }
}

}  // namespace

cudaError_t launch_quantize_tokens(const void *x, int64_t M, int64_t K, int64_t ldx, int bits, void *q, int fmt,
                                   float *s_tok, cudaStream_t st) {
    if (M == 0) return cudaSuccess;
    const int qmax = (1 << (bits - 1)) - 1;
    if (fmt == OT_CODE_F16)
        quantize_tokens_kernel<true><<<(unsigned)M, 256, 0, st>>>(reinterpret_cast<const __half *>(x), K, ldx, qmax,
                                                                  q, s_tok);
    else
        quantize_tokens_kernel<false><<<(unsigned)M, 256, 0, st>>>(reinterpret_cast<const __half *>(x), K, ldx,
                                                                   qmax, q, s_tok);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const void *x, int64_t M, int64_t K, int64_t ldx, const float *z, const float *r,
                            int bits, void *q, int fmt, cudaStream_t st, int32_t *rowsum) {
    if (M == 0) return cudaSuccess;
    const int qmax = (1 << (bits - 1)) - 1;
    dim3 grid((unsigned)((K + 255) / 256), (unsigned)((M + kQRowsPerBlock - 1) / kQRowsPerBlock));
    const __half *xh = reinterpret_cast<const __half *>(x);
    if (rowsum) {
        cudaError_t e = cudaMemsetAsync(rowsum, 0, (size_t)M * sizeof(int32_t), st);
        if (e != cudaSuccess) return e;
        if (fmt == OT_CODE_F16)
            quantize_kernel<true, true><<<grid, 256, 0, st>>>(xh, M, K, ldx, z, r, qmax, q, rowsum);
        else
            quantize_kernel<false, true><<<grid, 256, 0, st>>>(xh, M, K, ldx, z, r, qmax, q, rowsum);
    } else if (fmt == OT_CODE_F16) {
        return launch_kernel(quantize_kernel<true, false>, grid, dim3(256), 0, st, true, xh, M, K, ldx, z, r, qmax, q,
                             (int32_t *)nullptr);
    } else {
        return launch_kernel(quantize_kernel<false, false>, grid, dim3(256), 0, st, true, xh, M, K, ldx, z, r, qmax, q,
                             (int32_t *)nullptr);
    }
    return cudaGetLastError();
}

}  // namespace ot
