// gemv.cu -- the quantized linear of Eq. 6 / Eq. 7 for decode-sized token
// counts (M <= 32), where the product is bound by reading the int8 weights
// from HBM (each weight byte is used by only M tokens).
//
// A 128-row tcgen05 MMA costs about 118 cycles whatever its token count, which
// caps weight consumption at ~17 bytes per clock per SM (~5 TB/s on GB300),
// below the HBM rate.  Warp-level mma.sync m16n8k16 (f16 in, f32 accumulate)
// has throughput to spare at M <= 32 (600 TFLOPS measured), so here:
//   - a CTA of 16 (one token group) or 8 (two) warps owns 32 weight rows
//     (4 groups of 8 = the MMA's n8) and all tokens (groups of 16 = the MMA's
//     m16); the warps split K in interleaved 64-wide windows, issue the loads
//     of two windows before computing either (bytes in flight to cover HBM
//     latency), and reduce their int32 partial sums in shared memory at the
//     end (no global scratch);
//   - lane l of a warp loads 16 contiguous int8 weights of row (8g + l/4) at
//     K offset 16 (l % 4) of the window, widens them to fp16 in registers
//     (exact), and uses them as the MMA's B fragment under a fixed
//     permutation of K (the dot product does not depend on the order of k,
//     only on A and B using the same one): logical k {2t, 2t+1, 2t+8, 2t+9}
//     of lane-quad position t = l % 4 is actual K {16t+4j .. 16t+4j+3} in
//     sub-step j; the fp16 activation codes are read as the A fragment under
//     the same permutation;
//   - fp32 partial sums stay exact below 2^24 (chunks of kcb windows, as in
//     the tensor-memory kernels) and are added in int32.
#include <cuda_fp16.h>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

namespace {

constexpr int kGvRows = 32;   // weight rows per CTA
constexpr int kGvWin = 64;    // K per window
constexpr int kGvUnroll = 2;  // windows whose loads a warp issues before computing
// warps per CTA: 16 for one token group, 8 for two (register budget)
template <int TG>
__host__ __device__ constexpr int gv_warps() { return TG == 1 ? 16 : 8; }

__device__ __forceinline__ void i8x4_to_f16x4_gv(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t u = w ^ 0x80808080u;
    const uint32_t a = __byte_perm(u, 0x64646464u, 0x4140);
    const uint32_t b = __byte_perm(u, 0x64646464u, 0x4342);
    const __half2 bias = __half2half2(__ushort_as_half(0x6480));  // 1152
    const __half2 ha = __hsub2(*reinterpret_cast<const __half2 *>(&a), bias);
    const __half2 hb = __hsub2(*reinterpret_cast<const __half2 *>(&b), bias);
    lo = *reinterpret_cast<const uint32_t *>(&ha);
    hi = *reinterpret_cast<const uint32_t *>(&hb);
}

__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int TG, bool kS32>
__global__ void __launch_bounds__(gv_warps<TG>() * 32, 1) linear_gemv_kernel(const __half *__restrict__ q,
                                                                    const int8_t *__restrict__ qw,
                                                                    const float *__restrict__ sw,
                                                                    const float *__restrict__ bfold,
                                                                    void *__restrict__ out, int M, int N, int K,
                                                                    int ldy, int kcb, int relu,
                                                                    const float *__restrict__ s_tok) {
    constexpr int kGvWarps = gv_warps<TG>();
    __shared__ int32_t red[kGvWarps][TG * 16][kGvRows + 1];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = blockIdx.x * kGvRows;
    const int t = lane & 3, r = lane >> 2;
    const int nwin = (K + kGvWin - 1) / kGvWin;

    // weight rows of this lane (one per group of 8), clamped for the N tail
    const int8_t *wrow[4];
    bool wok[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        const int n = n0 + 8 * g + r;
        wok[g] = n < N;
        wrow[g] = qw + (int64_t)(wok[g] ? n : 0) * K;
    }
    // token rows of this lane: r and r + 8 of each token group
    const __half *qrow[TG][2];
    bool qok[TG][2];
#pragma unroll
    for (int tg = 0; tg < TG; ++tg)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int m = tg * 16 + r + 8 * h;
            qok[tg][h] = m < M;
            qrow[tg][h] = q + (int64_t)(qok[tg][h] ? m : 0) * K;
        }

    int32_t tot[TG][4][4];
    float acc[TG][4][4];
#pragma unroll
    for (int tg = 0; tg < TG; ++tg)
#pragma unroll
        for (int g = 0; g < 4; ++g)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                tot[tg][g][i] = 0;
                acc[tg][g][i] = 0.f;
            }

    int in_chunk = 0;
    for (int win0 = warp; win0 < nwin; win0 += kGvUnroll * kGvWarps) {
        uint4 wv[kGvUnroll][4];
        uint4 qv[kGvUnroll][TG][2][2];
        bool vok[kGvUnroll];
#pragma unroll
        for (int u = 0; u < kGvUnroll; ++u) {
            const int win = win0 + u * kGvWarps;
            const int k0 = win * kGvWin + 16 * t;  // this lane's 16 K of the window
            vok[u] = win < nwin;
            const bool kok = vok[u] && k0 < K;     // K % 16 == 0: a segment is whole or absent
#pragma unroll
            for (int g = 0; g < 4; ++g)
                wv[u][g] = (kok && wok[g]) ? __ldcs(reinterpret_cast<const uint4 *>(wrow[g] + k0))
                                           : make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int tg = 0; tg < TG; ++tg)
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int p = 0; p < 2; ++p)
                        qv[u][tg][h][p] = (kok && qok[tg][h])
                                              ? __ldg(reinterpret_cast<const uint4 *>(qrow[tg][h] + k0 + 8 * p))
                                              : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < kGvUnroll; ++u) {
            if (!vok[u]) break;
#pragma unroll
            for (int g = 0; g < 4; ++g) {
                uint32_t b[8];
                i8x4_to_f16x4_gv(wv[u][g].x, b[0], b[1]);
                i8x4_to_f16x4_gv(wv[u][g].y, b[2], b[3]);
                i8x4_to_f16x4_gv(wv[u][g].z, b[4], b[5]);
                i8x4_to_f16x4_gv(wv[u][g].w, b[6], b[7]);
#pragma unroll
                for (int tg = 0; tg < TG; ++tg) {
                    const uint32_t *x0 = reinterpret_cast<const uint32_t *>(&qv[u][tg][0][0]);  // token r
                    const uint32_t *x1 = reinterpret_cast<const uint32_t *>(&qv[u][tg][1][0]);  // token r + 8
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        // sub-step j covers actual K 16t + 4j .. 16t + 4j + 3 of the window
                        const uint32_t a[4] = {x0[2 * j], x1[2 * j], x0[2 * j + 1], x1[2 * j + 1]};
                        mma_16816(acc[tg][g], a, b[2 * j], b[2 * j + 1]);
                    }
                }
            }
            if (++in_chunk == kcb) {
                in_chunk = 0;
#pragma unroll
                for (int tg = 0; tg < TG; ++tg)
#pragma unroll
                    for (int g = 0; g < 4; ++g)
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            tot[tg][g][i] += __float2int_rn(acc[tg][g][i]);
                            acc[tg][g][i] = 0.f;
                        }
            }
        }
    }
#pragma unroll
    for (int tg = 0; tg < TG; ++tg)
#pragma unroll
        for (int g = 0; g < 4; ++g)
#pragma unroll
            for (int i = 0; i < 4; ++i) tot[tg][g][i] += __float2int_rn(acc[tg][g][i]);

    // accumulator fragment: c0 = (token r, row 2t), c1 = (r, 2t+1), c2 = (r+8, 2t), c3 = (r+8, 2t+1)
#pragma unroll
    for (int tg = 0; tg < TG; ++tg)
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            red[warp][tg * 16 + r][8 * g + 2 * t] = tot[tg][g][0];
            red[warp][tg * 16 + r][8 * g + 2 * t + 1] = tot[tg][g][1];
            red[warp][tg * 16 + r + 8][8 * g + 2 * t] = tot[tg][g][2];
            red[warp][tg * 16 + r + 8][8 * g + 2 * t + 1] = tot[tg][g][3];
        }
    __syncthreads();
    for (int idx = threadIdx.x; idx < TG * 16 * kGvRows; idx += kGvWarps * 32) {
        const int m = idx / kGvRows, c = idx % kGvRows;
        const int n = n0 + c;
        if (m >= M || n >= N) continue;
        int32_t s = 0;
#pragma unroll
        for (int w = 0; w < kGvWarps; ++w) s += red[w][m][c];
        if constexpr (kS32) {
            reinterpret_cast<int32_t *>(out)[(int64_t)m * N + n] = s;
        } else {
            const float scale = __ldg(sw + n);
            const float sc = s_tok ? __fmul_rn(__ldg(s_tok + m), scale) : scale;  // per-token path (Eq. 3)
            float v = __fmaf_rn(__int2float_rn(s), sc, __ldg(bfold + n));
            if (relu) v = fmaxf(v, 0.f);
            reinterpret_cast<__half *>(out)[(int64_t)m * ldy + n] = __float2half_rn(v);
        }
    }
}

template <int TG, bool kS32>
cudaError_t run_gemv(const LinearArgs &a, int kcb, cudaStream_t st) {
    const int grid = (int)((a.N + kGvRows - 1) / kGvRows);
    linear_gemv_kernel<TG, kS32><<<grid, gv_warps<TG>() * 32, 0, st>>>(
        reinterpret_cast<const __half *>(a.q), a.qw, a.sw, a.bfold, a.out, (int)a.M, (int)a.N, (int)a.K, (int)a.ldy,
        kcb, a.relu, a.s_tok);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_linear_gemv(const LinearArgs &a, int kcb, cudaStream_t st) {
    if (a.M <= 16) return a.out_s32 ? run_gemv<1, true>(a, kcb, st) : run_gemv<1, false>(a, kcb, st);
    return a.out_s32 ? run_gemv<2, true>(a, kcb, st) : run_gemv<2, false>(a, kcb, st);
}

}  // namespace ot
