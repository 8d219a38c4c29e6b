// gemv.cu -- the quantized linear of Eq. 6 / Eq. 7 for decode-sized token
// counts (M <= 16), where the product is bound by reading the int8 weights
// from HBM (each weight byte is used by only M tokens).
//
// At a few tokens a tcgen05 tile wastes most of its N width and its k-loop
// is bound by its barrier hand-offs; warp-level mma.sync m16n8k16 (f16 in,
// f32 accumulate) has throughput to spare, so the kernel is a weight stream
// (measured on GB300, OPT-13B QKV and fc2 shapes: faster than the tcgen05
// kernel up to 16 tokens, slower from 17):
//   - work units are (tile of 128 weight rows, 256-wide K slice); one
//     persistent CTA per SM takes a contiguous range of units, an equal share
//     of all of them (stream-K), so every SM streams the same number of bytes;
//   - each unit arrives in a ring of shared-memory stages as three TMA boxes:
//     two of 128 weight rows x 128 int8 (16 KB each, 128-byte swizzle,
//     evict-first: read once) and one of M tokens x 256 fp16 codes
//     (evict-last: every tile reads them again).  The tensor
//     maps zero-fill rows past N and K past the end, so ragged tails need no
//     special case.  Measured on GB300, the TMA unit of an SM completes about
//     one box per 176 ns whatever its size up to 8 KB, so boxes must be large:
//     8 KB boxes held the stream near 2.5 TB/s, 32 KB boxes reach ~7 TB/s;
//   - the first S units are issued at start; a producer warp (warp 16) then
//     refills each slot with the unit S places later as soon as the 16
//     consumer warps have arrived on the slot's empty barrier.  Measured on
//     GB300 (OPT-13B QKV / fc2, 1 token): 15.0 / 20.5 us against 17.3 / 23.1
//     with the refill issued by the last consumer warp done with the slot,
//     which then lagged behind the others and tended to be last again;
//   - the weights are the MMA's m16 operand and the tokens its n8 operand
//     (ceil(M / 8) token groups): warp w takes the 64-wide window w % 4 of
//     every stage and weight rows 32 (w / 4) .. + 31 (two m16 groups).  Lane l
//     reads 16 int8 weights of rows 16g + l/4 and 16g + l/4 + 8 at window
//     offset 16 (l % 4) and widens them to fp16 (exact) straight into A
//     fragment order, under a fixed permutation of K (the dot product does not
//     depend on the order of k, only on A and B using the same one): logical k
//     {2t, 2t+1, 2t+8, 2t+9} of lane-quad position t = l % 4 is actual K
//     {16t+4j .. 16t+4j+3} in sub-step j; the token codes, read under the same
//     permutation, are already the B fragment (two consecutive words);
//   - fp32 partial sums stay exact below 2^24 (chunks of kcb windows, as in
//     the tensor-memory kernels) and are added, as int32, into the tile's
//     totals in shared memory (atomics);
//   - a tile split between CTAs is finished by the CTA holding its first
//     unit, which works on it last (at the end of its range); the others work
//     on it first (at the start of theirs), store their int32 partials in a
//     workspace slot of their own and publish it with a launch-epoch flag
//     (release).  The finisher adds the slots (acquire; normally published
//     long before) and applies the epilogue.  The epoch is a counter in the
//     workspace: every launch takes counter + 1 and its last CTA stores that
//     back, so epochs grow from launch to launch (graph replays included), a
//     flag left by an earlier launch never matches and nothing has to be
//     cleared.
// Without a workspace the ranges are whole tiles (no split, less even).
#include <cuda_fp16.h>

#include <mutex>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

OT_DEBUG_UNIT(gemv)

namespace {

constexpr int kGvRows = 128;                      // weight rows per tile (16 MMA n8 groups)
constexpr int kGvKS = 256;                        // K per unit / stage (= the TMA box width)
constexpr int kGvWin = 64;                        // K per MMA window
constexpr int kGvWindows = kGvKS / kGvWin;        // windows per stage (4)
constexpr int kGvWarps = 16;
constexpr int kGvThreads = kGvWarps * 32;            // consumer threads (+ one producer warp)
constexpr int kGvWBox = kGvRows * 128;           // weight box: 128 rows x 128 bytes, 128-byte swizzle
constexpr int kGvWBytes = 2 * kGvWBox;            // weights of a stage (two boxes)
constexpr int kGvMaxStages = 8;
constexpr int kGvSmemBudget = 224 * 1024;
constexpr int kGvHeader = 384;                    // barriers, counters, flags
// Token box of a stage: fp16 codes (kGvF16) as copied; int8 codes (kGvI8),
// widened when the fragments are read; or fp16 activations (kGvX) that the
// CTA's warps quantize in place (z, r per channel) before any warp reads them.
constexpr int kGvF16 = 0, kGvI8 = 1, kGvX = 2;
constexpr int kGvPdlUnits = 2;                    // units whose weights load before a programmatic wait
constexpr int kGvSlotInts = kGvRows * 32;         // workspace ints per split tile (32 tokens x 128 rows)

struct GvParams {
    const float *sw, *bfold, *s_tok;
    const int32_t *zc, *rowsum;    // asymmetric weights: zero points [N], code row sums [M] (or null)
    const float *zq, *rq;          // chained epilogue: the next layer's z', r' [N] (or null)
    int qmax_out;
    void *out;
    int32_t *part;                 // [grid][kGvSlotInts] partial sums of split tiles (stream-K), or null
    unsigned long long *flags;     // [grid] launch epoch once a CTA's slot is complete
    unsigned long long *ctl;       // {epoch of the last launch, CTAs done with this one}
    int pdl;                       // launched as a programmatic dependent of the kernel before it
    int weights_early;             // that kernel is this call's quantize kernel: weights may load before it ends
    const float *xz, *xr;          // kGvX: z, r [K]
    int qmax_in;                   // kGvX: qmax of the codes
    int *status;        // device status word
    int M, N, K, ldy, kcb, relu;
    int nks;            // units per tile
    int stages, stage_bytes, red_bytes;
    int64_t ntiles, units;
    int grid;
    int whole;          // ranges of whole tiles (no workspace)
};

__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// First unit of CTA c's range.
__device__ __forceinline__ int64_t unit_begin(int64_t c, const GvParams &p) {
    if (p.whole) return c * p.ntiles / p.grid * p.nks;
    return c * p.units / p.grid;
}

// The CTA whose range holds unit x (ranges begin at floor(c * units / grid)):
// the largest c with c * units < (x + 1) * grid.
__device__ __forceinline__ int cta_of_unit(int64_t x, const GvParams &p) {
    return (int)(((x + 1) * p.grid + p.units - 1) / p.units - 1);
}

__device__ __forceinline__ uint64_t ld_acquire_flag(const unsigned long long *f) {
    uint64_t v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(f) : "memory");
    return v;
}

template <bool kS32>
__device__ __forceinline__ void store_out(const GvParams &p, int m, int n, int32_t s) {
    if constexpr (kS32) {
        if (OT_DCHECK(m < p.M && n < p.N)) reinterpret_cast<int32_t *>(p.out)[(int64_t)m * p.N + n] = s;
    } else {
        const float scale = __ldg(p.sw + n);
        const float sc = p.s_tok ? __fmul_rn(__ldg(p.s_tok + m), scale) : scale;  // per-token path (Eq. 3)
        // asymmetric weights: sum_k q (qw - zc_n) = acc - zc_n * rowsum_m; the entry point
        // bounds it below 2^31, so int32 arithmetic (wrapping in between) gives it exactly
        const float a = __int2float_rn(
            p.zc ? (int32_t)((uint32_t)s - (uint32_t)__ldg(p.zc + n) * (uint32_t)__ldg(p.rowsum + m)) : s);
        float v = __fmaf_rn(a, sc, __ldg(p.bfold + n));
        if (p.relu) v = fmaxf(v, 0.f);
        __half o;
        if (p.zq) {  // the next layer's code round((v - z') * r'), as an fp16 integer
            const int c = __float2int_rn(__fmul_rn(__fsub_rn(v, __ldg(p.zq + n)), __ldg(p.rq + n)));
            o = __int2half_rn(max(-p.qmax_out, min(p.qmax_out, c)));
        } else {
            o = __float2half_rn(v);
        }
        if (OT_DCHECK(m < p.M && n < p.N && p.N <= p.ldy))
            reinterpret_cast<__half *>(p.out)[(int64_t)m * p.ldy + n] = o;
    }
}

// Named barrier 1 over the 16 consumer warps (the producer warp takes no part).
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kGvThreads) : "memory"); }

// TN token groups of 8 (the MMA's n8); kTokG: the token box's format.
template <int TN, bool kS32, int kTokG>
__global__ void __launch_bounds__(kGvThreads + 32, 1)
    linear_gemv_kernel(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_a,
                       const GvParams p) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment: the swizzle pattern of a TMA box repeats every 1024 bytes
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(base);
    unsigned *loads = reinterpret_cast<unsigned *>(full + kGvMaxStages);  // units loaded into a slot, ever
    volatile int *abort = reinterpret_cast<volatile int *>(loads + kGvMaxStages);
    unsigned long long *epoch_s = reinterpret_cast<unsigned long long *>(base + 192);  // this launch's epoch
    uint64_t *qready = reinterpret_cast<uint64_t *>(base + 256);  // kGvX: the slot's codes are quantized
    uint64_t *empty = reinterpret_cast<uint64_t *>(base + 320);   // the 16 consumer warps are done with the slot
    int32_t(*red)[kGvRows + 1] = reinterpret_cast<int32_t(*)[kGvRows + 1]>(base + kGvHeader);  // [TN*8]
    uint8_t *ring = base + ((kGvHeader + p.red_bytes + 1023) & ~1023);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = p.stages;
    const int64_t u_begin = unit_begin(blockIdx.x, p), u_end = unit_begin(blockIdx.x + 1, p);
    const int M = p.M, N = p.N, K = p.K, nks = p.nks;
    const int64_t tile0 = u_begin / nks;
    const int ks0 = (int)(u_begin - tile0 * nks);
    const uint32_t abytes = (uint32_t)M * kGvKS * (kTokG == kGvI8 ? 1 : 2);  // token box
    uint64_t pol_w = 0, pol_a = 0;

    // Load unit (tile, ks) into `slot`, completing on full[slot]: the weight
    // boxes, then (load_codes) the codes box.
    // kGvX: the slice's z and r follow the activation box (channels below K only)
    const uint32_t zr_off = kGvWBytes + abytes;
    auto zr_bytes = [&](int ks) -> uint32_t {
        return kTokG == kGvX ? (uint32_t)min(kGvKS, K - ks * kGvKS) * 4 : 0u;
    };
    auto load_weights = [&](int slot, int64_t tile, int ks) {
        const uint32_t bar = smem_u32(&full[slot]);
        mbar_arrive_expect_tx(bar, kGvWBytes + abytes + 2 * zr_bytes(ks));
        const uint32_t st = smem_u32(ring + (size_t)slot * p.stage_bytes);
        tma_load_2d_hint(st, &tm_w, bar, ks * kGvKS, (int32_t)(tile * kGvRows), pol_w);
        tma_load_2d_hint(st + kGvWBox, &tm_w, bar, ks * kGvKS + 128, (int32_t)(tile * kGvRows), pol_w);
        loads[slot] += 1;
    };
    auto load_codes = [&](int slot, int ks) {
        const uint32_t st = smem_u32(ring + (size_t)slot * p.stage_bytes);
        tma_load_2d_hint(st + kGvWBytes, &tm_a, smem_u32(&full[slot]), ks * kGvKS, 0, pol_a);
        if constexpr (kTokG == kGvX) {
            bulk_load(st + zr_off, p.xz + ks * kGvKS, zr_bytes(ks), smem_u32(&full[slot]));
            bulk_load(st + zr_off + kGvKS * 4, p.xr + ks * kGvKS, zr_bytes(ks), smem_u32(&full[slot]));
        }
    };
    auto load_unit = [&](int slot, int64_t tile, int ks) {
        load_weights(slot, tile, ks);
        load_codes(slot, ks);
    };

    if (lane == 0) {
        pol_w = l2_policy_evict_first();
        pol_a = l2_policy_evict_last();
    }
    for (int i = threadIdx.x; i < TN * 8 * (kGvRows + 1); i += blockDim.x) (&red[0][0])[i] = 0;
    if (threadIdx.x == 0) {
        tma_prefetch_desc(&tm_w);
        tma_prefetch_desc(&tm_a);
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&qready[s]), kGvWarps);
            mbar_init(smem_u32(&empty[s]), kGvWarps);
            loads[s] = 0;
        }
        *abort = 0;
        fence_barrier_init();
        // Launched as a programmatic dependent, the kernel before this one on
        // the stream may still be running until grid_dep_wait() returns; until
        // then only the first units' weights are touched: loaded into the ring
        // when that kernel is this call's own quantize kernel (weights_early:
        // it lets this one start only after every earlier kernel, any writer
        // of the weights, has completed), else
        // prefetched into L2, which stays coherent with any write that kernel
        // makes.  The codes and the workspace are read only after the wait.
        // Without such a launch the loads go out unit by unit, so that the
        // first unit completes first.
        const int pre = p.weights_early ? (S < kGvPdlUnits ? S : kGvPdlUnits) : 0;
        int64_t tile = tile0;
        int ks = ks0;
        for (int s = 0; s < pre && u_begin + s < u_end; ++s) {
            load_weights(s, tile, ks);
            if (++ks == nks) {
                ks = 0;
                ++tile;
            }
        }
        if (p.pdl && !p.weights_early) {
            int64_t t2 = tile0;
            int k2 = ks0;
            for (int s = 0; s < S && u_begin + s < u_end; ++s) {
                tma_prefetch_l2_2d(&tm_w, k2 * kGvKS, (int32_t)(t2 * kGvRows));
                tma_prefetch_l2_2d(&tm_w, k2 * kGvKS + 128, (int32_t)(t2 * kGvRows));
                if (++k2 == nks) {
                    k2 = 0;
                    ++t2;
                }
            }
        }
        grid_dep_wait();
        *epoch_s = p.whole ? 0 : __ldcg(p.ctl) + 1;
        for (int s = 0, k2 = ks0; s < pre && u_begin + s < u_end; ++s) {
            load_codes(s, k2);
            if (++k2 == nks) k2 = 0;
        }
        for (int s = pre; s < S && u_begin + s < u_end; ++s) {
            load_unit(s, tile, ks);
            if (++ks == nks) {
                ks = 0;
                ++tile;
            }
        }
    }
    __syncthreads();
    // the next linear on the stream may launch now (it waits for this one before reading anything this writes)
    grid_dep_launch();
    if (warp == kGvWarps) {
        // producer warp: refills each slot with the unit S places later once
        // the 16 consumer warps are done with it
        if (lane == 0) {
            int64_t tile = tile0;
            int ks = ks0 + S;
            while (ks >= nks) {
                ks -= nks;
                ++tile;
            }
            for (int64_t i = S; u_begin + i < u_end; ++i) {
                const int slot = (int)(i % S);
                if (!mbar_wait(smem_u32(&empty[slot]), ((uint32_t)(i / S) & 1) ^ 1, abort, p.status)) break;
                load_unit(slot, tile, ks);
                if (++ks == nks) {
                    ks = 0;
                    ++tile;
                }
            }
            // teardown: every copy issued must land before the CTA's shared memory goes away
            for (int s2 = 0; s2 < S; ++s2)
                if (loads[s2] > 0) wait_teardown_status(smem_u32(&full[s2]), (loads[s2] - 1) & 1, p.status);
        }
        return;
    }

    const int t = lane & 3, r = lane >> 2;
    const int win = warp % kGvWindows, rp = warp / kGvWindows;  // window; rows 32 rp .. 32 rp + 31
    const int kw = win * kGvWin;
    bool tok[TN];  // this lane's token (8 tn + r) exists
    bool tgv[TN];  // some lane's does (warp-uniform)
#pragma unroll
    for (int tn = 0; tn < TN; ++tn) {
        tok[tn] = tn * 8 + r < M;
        tgv[tn] = tn * 8 < M;
    }
    // byte offsets inside a stage: this lane's weight row 32 rp + r and token row r
    // Lane r holds the A fragment rows r and r + 8 of each m16 group; logical row
    // r is the group's physical row sg = r/2 + 4 (r % 2), so that the two rows of
    // a quarter-warp (r = 2q, 2q + 1) sit 4 rows apart and their 128-byte
    // swizzles (16-byte chunk c stored at c ^ (row % 8)) fall in different bank halves.
    const int sg = (r >> 1) + 4 * (r & 1);
    const int w_off = (kw >> 7) * kGvWBox + (32 * rp + sg) * 128 + ((((kw & 127) >> 4) + t) ^ sg) * 16;
    constexpr int kEl = kTokG == kGvI8 ? 1 : 2;  // bytes per token value in the box
    const int a_off = kGvWBytes + r * (kEl * kGvKS) + kEl * (kw + 16 * t);

    float acc[2][TN][4];
#pragma unroll
    for (int g = 0; g < 2; ++g)
#pragma unroll
        for (int tn = 0; tn < TN; ++tn)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[g][tn][i] = 0.f;
    // Add the exact fp32 chunk sums into the tile's int32 totals in shared
    // memory.  Accumulator fragment: c0 = (row r, token 2t), c1 = (r, 2t+1),
    // c2 = (r+8, 2t), c3 = (r+8, 2t+1).
    auto flush = [&]() {
#pragma unroll
        for (int g = 0; g < 2; ++g)
#pragma unroll
            for (int tn = 0; tn < TN; ++tn)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int m = tn * 8 + 2 * t + (i & 1);
                    if (m < M) atomicAdd(&red[m][32 * rp + 16 * g + sg + 8 * (i >> 1)], __float2int_rn(acc[g][tn][i]));
                    acc[g][tn][i] = 0.f;
                }
    };

    int slot = 0;
    uint32_t phase = 0;
    int in_chunk = 0;
    int64_t tile = tile0;
    int ks = ks0;
    int64_t u = u_begin;
    while (u < u_end) {
        const int64_t seg_begin = u, seg_end = min(u_end, u + (nks - ks));
        const int mine = (int)(seg_end - u);
        for (; u < seg_end; ++u, ++ks) {
            bool ok;
            if constexpr (kTokG == kGvX) {
                // thread j quantizes the 16-byte chunk j (8 channels of one token) of the
                // box with the slice's z, r copied beside it; channels past K get code 0
                const int j = threadIdx.x;
                ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&full[slot]), phase, abort, p.status));
                if (ok && j < M * 32) {
                    uint8_t *stg = ring + (size_t)slot * p.stage_bytes;
                    float4 z0 = make_float4(0.f, 0.f, 0.f, 0.f), z1 = z0, q0 = z0, q1 = z0;
                    if (ks * kGvKS + (j & 31) * 8 < K) {
                        const float4 *zp = reinterpret_cast<const float4 *>(stg + zr_off + (j & 31) * 32);
                        const float4 *rp = reinterpret_cast<const float4 *>(stg + zr_off + kGvKS * 4 + (j & 31) * 32);
                        z0 = zp[0];
                        z1 = zp[1];
                        q0 = rp[0];
                        q1 = rp[1];
                    }
                    float2 nz[4], rq[4];
                    nz[0] = make_float2(-z0.x, -z0.y); nz[1] = make_float2(-z0.z, -z0.w);
                    nz[2] = make_float2(-z1.x, -z1.y); nz[3] = make_float2(-z1.z, -z1.w);
                    rq[0] = make_float2(q0.x, q0.y); rq[1] = make_float2(q0.z, q0.w);
                    rq[2] = make_float2(q1.x, q1.y); rq[3] = make_float2(q1.z, q1.w);
                    uint4 *c = reinterpret_cast<uint4 *>(stg + kGvWBytes + (j >> 5) * (2 * kGvKS) + (j & 31) * 16);
                    *c = quantize_f16x8(*c, nz, rq, p.qmax_in);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&qready[slot]));
                ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&qready[slot]), phase, abort, p.status)) && ok;
            } else {
                ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&full[slot]), phase, abort, p.status));
            }
            // past K the boxes hold zeros; skip windows that lie wholly past it
            if (ok && kw < K - ks * kGvKS) {
                if (in_chunk == p.kcb) {
                    in_chunk = 0;
                    flush();
                }
                ++in_chunk;
                const uint8_t *st = ring + (size_t)slot * p.stage_bytes;
                uint4 wv[2][2];  // [group][row r / r + 8]
#pragma unroll
                for (int g = 0; g < 2; ++g)
#pragma unroll
                    for (int h = 0; h < 2; ++h)
                        wv[g][h] = *reinterpret_cast<const uint4 *>(st + w_off + (16 * g + 8 * h) * 128);
                uint32_t x[TN][8];  // token 8 tn + r, actual K 16t .. 16t + 15 of the window (fp16 pairs)
#pragma unroll
                for (int tn = 0; tn < TN; ++tn) {
                    uint4 lo = make_uint4(0, 0, 0, 0), hi = make_uint4(0, 0, 0, 0);
                    if (tgv[tn] && tok[tn]) {
                        if constexpr (kTokG == kGvI8) {
                            const uint4 v = *reinterpret_cast<const uint4 *>(st + a_off + tn * 8 * kGvKS);
                            lo = i8x8_to_f16x8(make_uint2(v.x, v.y));
                            hi = i8x8_to_f16x8(make_uint2(v.z, v.w));
                        } else {
                            lo = *reinterpret_cast<const uint4 *>(st + a_off + tn * 8 * (2 * kGvKS));
                            hi = *reinterpret_cast<const uint4 *>(st + a_off + tn * 8 * (2 * kGvKS) + 16);
                        }
                    }
                    x[tn][0] = lo.x; x[tn][1] = lo.y; x[tn][2] = lo.z; x[tn][3] = lo.w;
                    x[tn][4] = hi.x; x[tn][5] = hi.y; x[tn][6] = hi.z; x[tn][7] = hi.w;
                }
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                    // A fragment of sub-step j: {row r: k pair 0, row r+8: k pair 0, row r: pair 1, row r+8: pair 1}
                    uint32_t a[4][4];
                    const uint32_t w0[4] = {wv[g][0].x, wv[g][0].y, wv[g][0].z, wv[g][0].w};
                    const uint32_t w1[4] = {wv[g][1].x, wv[g][1].y, wv[g][1].z, wv[g][1].w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        i8x4_to_f16x4(w0[j], a[j][0], a[j][2]);
                        i8x4_to_f16x4(w1[j], a[j][1], a[j][3]);
                    }
#pragma unroll
                    for (int tn = 0; tn < TN; ++tn) {
                        if (!tgv[tn]) continue;
#pragma unroll
                        for (int j = 0; j < 4; ++j) mma_16816(acc[g][tn], a[j], x[tn][2 * j], x[tn][2 * j + 1]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&empty[slot]));
            if (++slot == S) {
                slot = 0;
                phase ^= 1;
            }
        }

        // ---- end of this CTA's part of the tile: add the warps' totals ----
        in_chunk = 0;
        flush();
        consumers_sync();
        const int n0 = (int)(tile * kGvRows);
        if (mine == nks) {
            for (int idx = threadIdx.x; idx < M * kGvRows; idx += kGvThreads) {
                const int m = idx / kGvRows, c = idx % kGvRows;
                const int32_t s = red[m][c];
                red[m][c] = 0;
                if (n0 + c < N) store_out<kS32>(p, m, n0 + c, s);
            }
        } else if (seg_begin != tile * nks) {
            // a later part of a tile that an earlier CTA finishes: publish it
            int32_t *part = p.part + (size_t)blockIdx.x * kGvSlotInts;
            const bool in_ws = OT_DCHECK((int)blockIdx.x < p.grid && M * kGvRows <= kGvSlotInts);
            for (int idx = threadIdx.x; idx < M * kGvRows; idx += kGvThreads) {
                const int m = idx / kGvRows, c = idx % kGvRows;
                if (in_ws) __stcg(part + idx, red[m][c]);
                red[m][c] = 0;
            }
            __threadfence();
            consumers_sync();
            if (threadIdx.x == 0) {
                __threadfence();
                atomicExch(p.flags + blockIdx.x, *epoch_s);
            }
        } else {
            // the first part: add the later parts (CTAs blockIdx.x + 1 .. last) and finish the tile
            const int c_last = cta_of_unit((tile + 1) * nks - 1, p);
            const int nc = c_last - (int)blockIdx.x;
            if (threadIdx.x < nc) {
                const unsigned long long *f = p.flags + blockIdx.x + 1 + threadIdx.x;
                const uint64_t t0 = globaltimer_ns();
                const unsigned long long epoch = *epoch_s;
                while (ld_acquire_flag(f) != epoch) {
                    if (*abort) break;
                    if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
                        atomicExch(p.status, (int)OT_ERR_TIMEOUT);
                        *abort = 1;
                        break;
                    }
                }
            }
            consumers_sync();
            for (int idx = threadIdx.x; idx < M * kGvRows; idx += kGvThreads) {
                const int m = idx / kGvRows, c = idx % kGvRows;
                int32_t s = red[m][c];
                red[m][c] = 0;
                for (int j = 1; j <= nc; ++j) s += __ldcg(p.part + (size_t)(blockIdx.x + j) * kGvSlotInts + idx);
                if (n0 + c < N) store_out<kS32>(p, m, n0 + c, s);
            }
        }
        consumers_sync();  // red is reused by the next tile
        ks = 0;
        ++tile;
    }
    // teardown (only matters after a timeout): every copy issued must land
    // before the CTA's shared memory goes away
    if (threadIdx.x == 0) {
        if (!p.whole && atomicAdd(p.ctl + 1, 1ull) == (unsigned long long)gridDim.x - 1) {
            // the last CTA of the launch: hand the epoch to the next launch
            p.ctl[1] = 0;
            p.ctl[0] = *epoch_s;
        }
    }
}

template <int TN, bool kS32, int kTokG>
cudaError_t run_gemv(const CUtensorMap &tm_w, const CUtensorMap &tm_a, const GvParams &base, cudaStream_t st,
                     bool pdl) {
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(linear_gemv_kernel<TN, kS32, kTokG>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, kGvSmemBudget);
    });
    if (attr_err != cudaSuccess) return attr_err;
    GvParams p = base;
    p.red_bytes = (TN * 8 * (kGvRows + 1) * 4 + 127) / 128 * 128;
    p.stage_bytes = (kGvWBytes + p.M * kGvKS * (kTokG == kGvI8 ? 1 : 2) + (kTokG == kGvX ? 2 * kGvKS * 4 : 0) + 1023) &
                    ~1023;
    const int ring_off = (kGvHeader + p.red_bytes + 1023) & ~1023;
    const int room = kGvSmemBudget - 1024 - ring_off;
    p.stages = room / p.stage_bytes;
    if (p.stages > kGvMaxStages) p.stages = kGvMaxStages;
    if (p.stages < 2) return cudaErrorInvalidConfiguration;
    const size_t smem = 1024 + ring_off + (size_t)p.stages * p.stage_bytes;
    return launch_kernel(linear_gemv_kernel<TN, kS32, kTokG>, dim3(p.grid), dim3(kGvThreads + 32), smem, st, pdl, tm_w,
                         tm_a, p);
}

}  // namespace

size_t gemv_workspace_bytes() {
    const size_t g = (size_t)num_sms();
    return g * kGvSlotInts * sizeof(int32_t) + g * sizeof(unsigned long long) + 2 * sizeof(unsigned long long);
}

cudaError_t launch_linear_gemv(const LinearArgs &a, int kcb, cudaStream_t st) {
    // weights: boxes of 128 rows x 128 int8 (128-byte swizzle); codes: boxes of
    // all M tokens x 256 fp16 (no swizzle); both zero-filled outside the arrays
    // (int8 codes: boxes of all M tokens x 256 int8; fp16 activations: rows of ldx elements)
    CUtensorMap tm_w, tm_a;
    const bool i8 = a.q_fmt == kCodesI8;
    const uint64_t arow = i8 ? (uint64_t)a.K : (uint64_t)(a.q_fmt == kActF16 ? a.ldx : a.K) * 2;
    if (!tensor_map_2d(&tm_w, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.qw, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K,
                       128, kGvRows, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !tensor_map_2d(&tm_a, i8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a.q,
                       (uint64_t)a.K, (uint64_t)a.M, arow, kGvKS, (uint32_t)a.M, CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorInvalidValue;
    GvParams p{};
    p.sw = a.sw;
    p.bfold = a.bfold;
    p.s_tok = a.s_tok;
    p.zc = a.zc;
    p.rowsum = a.rowsum;
    p.zq = a.zq;
    p.rq = a.rq;
    p.qmax_out = a.qmax_out;
    p.pdl = a.pdl ? 1 : 0;
    p.weights_early = a.pdl && a.weights_early ? 1 : 0;
    p.xz = a.xz;
    p.xr = a.xr;
    p.qmax_in = a.qmax_in;
    p.out = a.out;
    p.status = device_status_word();
    if (!p.status) return cudaErrorUnknown;
    p.M = (int)a.M;
    p.N = (int)a.N;
    p.K = (int)a.K;
    p.ldy = (int)a.ldy;
    p.kcb = kcb;
    p.relu = a.relu;
    p.nks = (int)((a.K + kGvKS - 1) / kGvKS);
    p.ntiles = (a.N + kGvRows - 1) / kGvRows;
    p.units = p.ntiles * p.nks;
    const int sms = num_sms();
    // a.workspace here is the decode region of the caller's workspace.  Split
    // tiles even out the per-SM work but add the partial-sum exchange, and the
    // weight stream saturates HBM once about 60% of the SMs take part; so whole
    // tiles are kept when they already occupy that many SMs and the busiest
    // CTA gets at most 25% more units than an even split would give it
    // (measured on GB300: OPT-13B QKV and 16384 x 4096 at one token run 8-15%
    // faster on whole tiles, fc2 and 4096 x 4096 2-2.5x faster split).
    const int64_t active = p.ntiles < sms ? p.ntiles : sms;
    const int64_t whole_units = (p.ntiles + sms - 1) / sms * p.nks;
    const int64_t even_units = (p.units + sms - 1) / sms;
    const bool whole_ok = 10 * active >= 6 * (int64_t)sms && 4 * whole_units <= 5 * even_units;
    const bool split = !whole_ok && a.workspace != nullptr && a.workspace_bytes >= gemv_workspace_bytes();
    if (split) {
        p.whole = 0;
        p.grid = (int)(p.units < sms ? p.units : sms);
        p.part = reinterpret_cast<int32_t *>(a.workspace);
        p.flags = reinterpret_cast<unsigned long long *>(p.part + (size_t)sms * kGvSlotInts);
        p.ctl = p.flags + sms;
    } else {
        p.whole = 1;
        p.grid = (int)(p.ntiles < sms ? p.ntiles : sms);
    }
    const bool d = a.pdl;
    if (a.M > 16) return cudaErrorInvalidValue;  // more than 16 tokens go to the tcgen05 kernels
    const bool one = a.M <= 8;
    if (a.q_fmt == kActF16)
        return one ? run_gemv<1, false, kGvX>(tm_w, tm_a, p, st, d) : run_gemv<2, false, kGvX>(tm_w, tm_a, p, st, d);
    if (i8) {
        if (a.out_s32)
            return one ? run_gemv<1, true, kGvI8>(tm_w, tm_a, p, st, d)
                       : run_gemv<2, true, kGvI8>(tm_w, tm_a, p, st, d);
        return one ? run_gemv<1, false, kGvI8>(tm_w, tm_a, p, st, d)
                   : run_gemv<2, false, kGvI8>(tm_w, tm_a, p, st, d);
    }
    if (a.out_s32)
        return one ? run_gemv<1, true, kGvF16>(tm_w, tm_a, p, st, d) : run_gemv<2, true, kGvF16>(tm_w, tm_a, p, st, d);
    return one ? run_gemv<1, false, kGvF16>(tm_w, tm_a, p, st, d) : run_gemv<2, false, kGvF16>(tm_w, tm_a, p, st, d);
}

}  // namespace ot
