// gemm.cu -- the quantized linear of Eq. 6 / Eq. 7 on sm_103a tensor cores:
//   acc[m,n] = sum_k q[m,k] * qw[n,k]           (exact integers)
//   y[m,n]   = fp16(fma((float)acc, sw_n, b'_n)) (+ ReLU)   or acc as int32
//
// sm_103a has no integer tcgen05.mma (kind::i8 is an sm_100a feature), so
// the product runs on tcgen05.mma kind::f16: integer codes |c| <= 127 are
// exact in fp16, every product is exact in fp32, and an fp32 sum of integers
// is exact while it stays below 2^24.  K is therefore summed in chunks of
// kcb k-blocks with kcb * 64 * qmax_a * qmax_w <= 2^24; each chunk's fp32
// accumulator is converted to int32 (exact) and summed in registers.
//
// Two kernels: linear_kernel (below; 16 < M <= 64, int8 codes and the
// in-producer quantization up to 128 tokens, and any M when K % 128 != 0) and
// linear_pair_kernel (K % 128 == 0 and M > 64: CTA pairs, 192-token tiles above
// 128 tokens, 128-token tiles for 65-128; its own comment further down).  The
// TMA and MMA roles of both run their loops with the whole warp and issue
// from one elected lane.
//
// linear_kernel (one persistent CTA per SM, 16 warps):
//   warp 0        TMA producer: per 64-wide k-block, the activation-code tile
//                 (BN tokens x 64, fp16, 128-byte swizzle) and the weight tile
//                 (128 rows x 64, int8, 64-byte swizzle) into a 6-stage ring.
//   warp 1        MMA issuer (one thread): D[128 x BN] += A[128 x 16] * B,
//                 A read from tensor memory, B from shared memory.
//   warp 2        allocates / frees the 512 TMEM columns.
//   warps 4-7     converters: each thread takes one weight row of the stage,
//                 turns its 64 int8 codes into fp16 pairs in registers and
//                 stores them into the TMEM A buffer of the stage
//                 (tcgen05.st), so the int8 -> fp16 widening never costs
//                 shared-memory bandwidth.
//   warps 8-15    epilogue: drain each finished chunk accumulator (double
//                 buffered in TMEM) into int32 totals, and at the end of the
//                 tile apply sw_n, b'_n, ReLU and store.
// The weight matrix is the MMA's M side (128 output channels = TMEM lanes),
// tokens are its N side (BN = 16..128), i.e. the kernel computes Y^T tiles.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "ot_common.cuh"
#include "ot_kernels.h"

namespace ot {

// Device status word of this library (OT_OK or OT_ERR_TIMEOUT), one per device.
__device__ int g_status;
OT_DEBUG_UNIT(gemm)

namespace {

constexpr int kBM = 128;        // weight rows per tile (TMEM lanes, MMA M)
constexpr int kBK = 64;         // K elements per k-block (128 bytes of fp16)
constexpr int kStages = 6;      // shared-memory ring and TMEM A buffers
constexpr int kThreads = 512;   // 16 warps
constexpr int kWarpTma = 0, kWarpMma = 1, kWarpAlloc = 2, kWarpConv0 = 4, kWarpEpi0 = 8;
constexpr int kNumEpiWarps = 8;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemAccCol = 256;   // A buffers at columns [0, 32*kStages), accumulators from 256
static_assert(32 * kStages <= (int)kTmemAccCol, "TMEM A buffers overlap the accumulators");

// Token operand of linear_kernel (its MMA's B): fp16 codes copied by TMA as
// they are (kTokF16); int8 codes copied into a staging buffer and widened to
// fp16 by four token warps (kTokI8); or fp16 activations copied by TMA and
// quantized in place by the token warps, per channel with z and r (kTokX:
// the quantization of Eq. 6 / Eq. 7 inside the GEMM's operand producer).
constexpr int kTokF16 = 0, kTokI8 = 1, kTokX = 2;
constexpr int kWarpTok0 = 16;  // token warps 16-19 (kTok != kTokF16: 20 warps)
template <int kTok>
__host__ __device__ constexpr int lin_threads() { return kTok == kTokF16 ? kThreads : kThreads + 128; }

template <int BN, int kTok>
struct alignas(1024) Smem {
    uint8_t b[kStages][BN * 128];   // activation codes, 128-byte swizzled rows
    uint8_t w[kStages][kBM * kBK];  // int8 weight codes, 64-byte swizzled rows
    uint8_t bs[kTok == kTokI8 ? kStages : 1][kTok == kTokI8 ? BN * 64 : 16];  // int8 codes as copied (kTokI8)
    alignas(16) float zr[kTok == kTokX ? kStages : 1][2][64];  // kTokX: the k-block's z and r, copied with the tiles
    uint64_t full[kStages];         // TMA landed (tx bytes)
    uint64_t empty[kStages];        // stage free: MMA done with b[] + 4 converter warps done with w[]
                                    // (+ kTokI8: 4 token warps done with bs[])
    uint64_t afull[kStages];        // TMEM A buffer written (4 converter warps)
    uint64_t aempty[kStages];       // TMEM A buffer consumed (MMA commit)
    uint64_t bfull[kStages];        // kTok != kTokF16: b[] holds fp16 codes (4 token warps)
    uint64_t accfull[2];            // chunk accumulator complete (MMA commit)
    uint64_t accempty[2];           // chunk accumulator drained (8 epilogue warps)
    uint64_t drain;                 // teardown: all issued MMAs complete
    uint64_t pub;                   // stream-K: the 8 epilogue warps stored their partial sums
    uint32_t tmem_base;
    int abort;
    unsigned long long epoch;       // stream-K: this launch's flag value
};

// Bounded wait that ignores the abort flag (used only while tearing down).
__device__ __forceinline__ void wait_teardown(uint32_t bar, uint32_t parity) {
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
            atomicExch(&g_status, (int)OT_ERR_TIMEOUT);
            return;
        }
    }
}

// Work of one worker (a CTA pair of linear_pair_kernel, a CTA of
// linear_kernel): a list of pieces (tile u, k-blocks [kb0, kb1)).
// Without a workspace the pieces are whole tiles dealt round-robin.  With a
// workspace (stream-K) all but the last full round of tiles are still dealt
// whole (neighbouring pairs then share weight and token tiles in L2), and
// the remaining tiles' flattened (tile, k-block) space is cut into equal
// contiguous ranges, one per pair, so no pair idles in a last partial round.
// A pair walks its stream-K tiles in reverse, so the piece that does not end
// a tile (its partial int32 sums go to the workspace) comes first and the
// piece that ends a tile (it adds the partials of the earlier pairs) last.
struct PairSched {
    int nkb, streamk, count;
    int first, stride, dp;      // whole tiles: u = first + p * stride for p < dp
    int sk0;                    // first stream-K tile
    int begin, end, u_last;     // this pair's stream-K range (flattened, relative to sk0)
    int per, rem;

    __device__ void init(int num_units, int nkb_, int nclusters, int cluster, bool use_streamk) {
        nkb = nkb_;
        streamk = use_streamk ? 1 : 0;
        first = cluster;
        stride = nclusters;
        if (!streamk) {
            dp = cluster < num_units ? (num_units - cluster + nclusters - 1) / nclusters : 0;
            count = dp;
            return;
        }
        const int rounds = num_units / nclusters;
        dp = rounds >= 2 ? rounds - 1 : 0;
        sk0 = dp * nclusters;
        const int total = (num_units - sk0) * nkb;
        const int active = total < nclusters ? total : nclusters;
        per = active > 0 ? total / active : 0;
        rem = active > 0 ? total % active : 0;
        count = dp;
        if (cluster >= active) return;
        begin = cluster * per + (cluster < rem ? cluster : rem);
        end = begin + per + (cluster < rem ? 1 : 0);
        u_last = (end - 1) / nkb;
        count += u_last - begin / nkb + 1;
    }
    __device__ void piece(int p, int &u, int &kb0, int &kb1) const {
        if (p < dp) {
            u = first + p * stride;
            kb0 = 0;
            kb1 = nkb;
            return;
        }
        const int v = u_last - (p - dp);  // stream-K tile, relative to sk0
        u = sk0 + v;
        kb0 = max(begin, v * nkb) - v * nkb;
        kb1 = min(end, (v + 1) * nkb) - v * nkb;
    }
    // the first pair whose stream-K range holds part of tile u
    __device__ int first_owner(int u) const {
        const int x = (u - sk0) * nkb;
        const int big = rem * (per + 1);
        return x < big ? x / (per + 1) : rem + (x - big) / per;
    }
};

// Order of the pair kernel's tiles (unit u -> token tile mt, weight-row pair np):
// groups of `group_m` token tiles, token tiles fastest within a group, so the
// clusters running at one time share few token tiles and a group's codes stay
// in L2 while the weight tiles stream past them once per group
// (group_m == m_tiles: the plain order, token tiles fastest).
__device__ __forceinline__ void pair_tile(int u, int m_tiles, int n_pairs, int group_m, int &mt, int &np) {
    const int per_group = group_m * n_pairs;
    const int g = u / per_group;
    const int first = g * group_m;
    const int size = min(group_m, m_tiles - first);
    const int r = u - g * per_group;
    mt = first + r % size;
    np = r / size;
}

// Stream-K workspace: per pair and CTA rank, 256 token columns x 128 weight
// rows of int32 partial sums (column-major, so a warp's stores are
// contiguous), then one 64-bit flag per pair and rank holding the launch
// epoch once its partials are complete, then the epoch counter and a count of
// the CTAs done with the launch.  Each launch takes epoch = counter + 1; the
// last CTA to finish stores it back (a launch starts only after the previous
// one on the stream ended, so all CTAs of a launch read one value), so the
// epochs grow from launch to launch on the device -- also when the launch is
// replayed from a CUDA graph -- and a flag left by an earlier launch never
// matches.  A zero-filled workspace starts the count.
__host__ __device__ constexpr size_t pair_slot_ints() { return (size_t)256 * 128; }

// {epoch of the last launch, CTAs done with this one}, after the flags
__device__ __forceinline__ unsigned long long *pair_ctl(int32_t *ws, int nclusters) {
    return reinterpret_cast<unsigned long long *>(ws + (size_t)nclusters * 2 * pair_slot_ints()) +
           (size_t)nclusters * 2;
}

__device__ __forceinline__ uint64_t ld_acquire_u64(const unsigned long long *p) {
    uint64_t v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

template <int BN, bool kS32, bool kAsym, bool kQOut, int kTok>
__global__ void __launch_bounds__(lin_threads<kTok>(), 1)
    linear_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_w,
                  const float *__restrict__ sw, const float *__restrict__ bfold, void *__restrict__ out, int M,
                  int N, int K, int ldy, int kcb, int relu, const float *__restrict__ s_tok,
                  const int32_t *__restrict__ zc, const int32_t *__restrict__ rowsum,
                  const float *__restrict__ zq, const float *__restrict__ rq, int qmax_out,
                  int32_t *__restrict__ ws, int ws_pairs, const float *__restrict__ xz,
                  const float *__restrict__ xr, int qmax_in) {
    extern __shared__ uint8_t smem_raw[];
    Smem<BN, kTok> &S =
        *reinterpret_cast<Smem<BN, kTok> *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = warp_id(), lane = lane_id();
    const int m_tiles = (M + BN - 1) / BN;
    const int n_tiles = (N + kBM - 1) / kBM;
    const int num_tiles = m_tiles * n_tiles;
    const int nkb = (K + kBK - 1) / kBK;
    volatile int *abort = &S.abort;
    constexpr uint32_t kTxBytes = (kTok == kTokI8 ? BN * 64 : BN * 128) + kBM * kBK;
    // With a workspace (the prefill kernel's layout, ws_pairs pairs of slots)
    // the CTAs split tiles along K like the pairs of linear_pair_kernel.
    PairSched sch;
    sch.init(num_tiles, nkb, gridDim.x, blockIdx.x, ws != nullptr);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&S.full[s]), 1);
            mbar_init(smem_u32(&S.empty[s]), 1 + 4 + (kTok == kTokI8 ? 4 : 0));
            mbar_init(smem_u32(&S.afull[s]), 4);
            mbar_init(smem_u32(&S.aempty[s]), 1);
            mbar_init(smem_u32(&S.bfull[s]), 4);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&S.accfull[b]), 1);
            mbar_init(smem_u32(&S.accempty[b]), kNumEpiWarps);
        }
        mbar_init(smem_u32(&S.drain), 1);
        mbar_init(smem_u32(&S.pub), kNumEpiWarps);
        S.abort = 0;
        fence_barrier_init();
        // Launched as a programmatic dependent, the kernel before this one may
        // still be running: prefetch the first weights into L2 (coherent with
        // any write it makes), then wait for it before anything reads the
        // codes or the workspace.
        if (sch.count > 0) {
            int u, pk0, pk1;
            sch.piece(0, u, pk0, pk1);
            for (int kb = pk0; kb < pk1 && kb < pk0 + kStages; ++kb)
                tma_prefetch_l2_2d(&tm_w, kb * kBK, (u / m_tiles) * kBM);
        }
        grid_dep_wait();
        S.epoch = ws ? __ldcg(pair_ctl(ws, ws_pairs)) + 1 : 0;
    }
    if (warp == kWarpTma && lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_w);
    }
    if (warp == kWarpAlloc) {
        tmem_alloc(smem_u32(&S.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    // the next linear on the stream may launch now (it waits for this one before reading anything this writes)
    grid_dep_launch();

    // the TMA and MMA roles run their loops with the whole warp and issue from one elected lane
    // registers: 512 threads x 128 at launch (kTokF16); with the token warps
    // 640 x 96, then per warpgroup 48 / 72 / 144 / 144 / 72
    if (warp < kWarpConv0) {
        if constexpr (kTok != kTokF16) regs_dec<48>();
        if (warp == kWarpTma) {
            uint32_t it = 0;
            bool ok = true;
            for (int p = 0; p < sch.count && ok; ++p) {
                int u, pk0, pk1;
                sch.piece(p, u, pk0, pk1);
                const int m0 = (u % m_tiles) * BN, n0 = (u / m_tiles) * kBM;
                for (int kb = pk0; kb < pk1; ++kb, ++it) {
                    const int s = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!(ok = mbar_wait_warp(smem_u32(&S.empty[s]), ph ^ 1, abort, &g_status))) break;
                    if (elect_one()) {
                        // kTokX: the k-block's z and r (channels below K only; K % 16 == 0, so the
                        // byte count stays a multiple of 64)
                        const uint32_t zr_bytes = kTok == kTokX ? (uint32_t)min(kBK, K - kb * kBK) * 4 : 0;
                        mbar_arrive_expect_tx(smem_u32(&S.full[s]), kTxBytes + 2 * zr_bytes);
                        tma_load_2d(smem_u32(kTok == kTokI8 ? S.bs[s % (kTok == kTokI8 ? kStages : 1)] : S.b[s]),
                                    &tm_q, smem_u32(&S.full[s]), kb * kBK, m0);
                        tma_load_2d(smem_u32(S.w[s]), &tm_w, smem_u32(&S.full[s]), kb * kBK, n0);
                        if constexpr (kTok == kTokX) {
                            const int zs = s % (kTok == kTokX ? kStages : 1);
                            bulk_load(smem_u32(S.zr[zs][0]), xz + kb * kBK, zr_bytes, smem_u32(&S.full[s]));
                            bulk_load(smem_u32(S.zr[zs][1]), xr + kb * kBK, zr_bytes, smem_u32(&S.full[s]));
                        }
                    }
                    __syncwarp();
                }
            }
            // teardown: every load issued must have landed before the CTA exits
            if (lane == 0) {
                const uint32_t issued = it;
                for (uint32_t j = issued > (uint32_t)kStages ? issued - kStages : 0; j < issued; ++j)
                    wait_teardown(smem_u32(&S.full[j % kStages]), (j / kStages) & 1);
            }
            __syncwarp();
        } else if (warp == kWarpMma) {
            const uint32_t idesc = idesc_f16_f32(kBM, BN);
            uint32_t it = 0, g = 0;
            bool ok = true;
            for (int p = 0; p < sch.count && ok; ++p) {
                int u, pk0, pk1;
                sch.piece(p, u, pk0, pk1);
                for (int kb0 = pk0; kb0 < pk1 && ok; kb0 += kcb, ++g) {
                    const int buf = g & 1;
                    if (!(ok = mbar_wait_warp(smem_u32(&S.accempty[buf]), ((g >> 1) & 1) ^ 1, abort, &g_status))) break;
                    tc_fence_after();
                    const uint32_t d = tmem + kTmemAccCol + buf * BN;
                    const int kb1 = min(pk1, kb0 + kcb);
                    for (int kb = kb0; kb < kb1; ++kb, ++it) {
                        const int s = it % kStages;
                        const uint32_t ph = (it / kStages) & 1;
                        // the token warps and the converters both start after the stage's copies landed
                        const uint32_t bbar = kTok == kTokF16 ? smem_u32(&S.full[s]) : smem_u32(&S.bfull[s]);
                        if (!(ok = mbar_wait_warp(bbar, ph, abort, &g_status))) break;
                        if (!(ok = mbar_wait_warp(smem_u32(&S.afull[s]), ph, abort, &g_status))) break;
                        tc_fence_after();
                        const uint64_t bdesc = smem_desc_sw128(smem_u32(S.b[s]));
                        if (elect_one()) {
    #pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk)
                                mma_f16_ts(d, tmem + s * 32 + kk * 8, bdesc + (uint64_t)((kk * 32) >> 4), idesc,
                                           (kb != kb0 || kk != 0) ? 1u : 0u);
                            mma_commit(smem_u32(&S.empty[s]));
                            mma_commit(smem_u32(&S.aempty[s]));
                        }
                        __syncwarp();
                    }
                    if (ok && elect_one()) mma_commit(smem_u32(&S.accfull[buf]));
                    __syncwarp();
                }
            }
            // teardown: all issued MMAs complete before TMEM is freed
            if (elect_one()) {
                mma_commit(smem_u32(&S.drain));
                wait_teardown(smem_u32(&S.drain), 0);
            }
            __syncwarp();
        }
    } else if (warp < kWarpEpi0) {
        if constexpr (kTok != kTokF16) regs_dec<72>();
        const int q = warp & 3;
        const int row = q * 32 + lane;           // weight row of the tile = TMEM lane
        const uint32_t sw64 = (row >> 1) & 3;    // 64-byte swizzle phase of this row
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t it = 0;
        bool ok = true;
        for (int p = 0; p < sch.count && ok; ++p) {
            int u, pk0, pk1;
            sch.piece(p, u, pk0, pk1);
            for (int kb = pk0; kb < pk1; ++kb, ++it) {
                const int s = it % kStages;
                const uint32_t ph = (it / kStages) & 1;
                if (!(ok = mbar_wait(smem_u32(&S.full[s]), ph, abort, &g_status))) break;
                uint4 raw[4];
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    raw[c] = *reinterpret_cast<const uint4 *>(S.w[s] + row * 64 + ((c ^ sw64) << 4));
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.empty[s]));
                // the row's 64 fp16 values, two per 32-bit TMEM column, k ascending; widened
                // before waiting for the TMEM buffer, so only the store follows the wait
                uint32_t a[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    i8x4_to_f16x4(raw[c].x, a[8 * c + 0], a[8 * c + 1]);
                    i8x4_to_f16x4(raw[c].y, a[8 * c + 2], a[8 * c + 3]);
                    i8x4_to_f16x4(raw[c].z, a[8 * c + 4], a[8 * c + 5]);
                    i8x4_to_f16x4(raw[c].w, a[8 * c + 6], a[8 * c + 7]);
                }
                if (!(ok = mbar_wait(smem_u32(&S.aempty[s]), ph ^ 1, abort, &g_status))) break;
                tc_fence_after();
                tmem_st32(tmem + lane_base + s * 32, a);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.afull[s]));
            }
        }
    } else if (kTok != kTokF16 && warp >= kWarpTok0) {
        if constexpr (kTok != kTokF16) regs_dec<72>();
        // token warps: thread t takes the 16-byte chunk cl (8 channels) of rows
        // r0, r0 + 16, ... of each k-block; r & 7 is the same for all of them,
        // so the chunk's place under the 128-byte swizzle, cl ^ (r & 7), is fixed
        const int t = (int)threadIdx.x - kWarpTok0 * 32;
        const int cl = t & 7, r0 = t >> 3;
        const int cp = (cl ^ (r0 & 7)) << 4;
        uint32_t it = 0;
        bool ok = true;
        for (int p = 0; p < sch.count && ok; ++p) {
            int u, pk0, pk1;
            sch.piece(p, u, pk0, pk1);
            for (int kb = pk0; kb < pk1; ++kb, ++it) {
                const int s = it % kStages;
                const uint32_t ph = (it / kStages) & 1;
                if (!(ok = mbar_wait(smem_u32(&S.full[s]), ph, abort, &g_status))) break;
                float2 nz[4], rr[4];
                if constexpr (kTok == kTokX) {
                    // channels past K (zero-filled by the copy; their z, r not copied) get z = r = 0: code 0
                    float4 z0 = make_float4(0.f, 0.f, 0.f, 0.f), z1 = z0, q0 = z0, q1 = z0;
                    if (kb * kBK + cl * 8 < K) {
                        const int zs = s % (kTok == kTokX ? kStages : 1);
                        const float4 *zp = reinterpret_cast<const float4 *>(S.zr[zs][0] + cl * 8);
                        const float4 *rp = reinterpret_cast<const float4 *>(S.zr[zs][1] + cl * 8);
                        z0 = zp[0];
                        z1 = zp[1];
                        q0 = rp[0];
                        q1 = rp[1];
                    }
                    nz[0] = make_float2(-z0.x, -z0.y); nz[1] = make_float2(-z0.z, -z0.w);
                    nz[2] = make_float2(-z1.x, -z1.y); nz[3] = make_float2(-z1.z, -z1.w);
                    rr[0] = make_float2(q0.x, q0.y); rr[1] = make_float2(q0.z, q0.w);
                    rr[2] = make_float2(q1.x, q1.y); rr[3] = make_float2(q1.z, q1.w);
                }
                uint8_t *bt = S.b[s] + cp;
                if constexpr (kTok == kTokI8) {
                    uint2 v[BN / 16];
#pragma unroll
                    for (int i = 0; i < BN / 16; ++i)
                        v[i] = *reinterpret_cast<const uint2 *>(S.bs[s % (kTok == kTokI8 ? kStages : 1)] +
                                                                (r0 + 16 * i) * 64 + cl * 8);
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&S.empty[s]));  // staging read
#pragma unroll
                    for (int i = 0; i < BN / 16; ++i)
                        *reinterpret_cast<uint4 *>(bt + (r0 + 16 * i) * 128) = i8x8_to_f16x8(v[i]);
                } else {
#pragma unroll
                    for (int i0 = 0; i0 < BN / 16; i0 += 4) {
                        uint4 v[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            v[i] = *reinterpret_cast<const uint4 *>(bt + (r0 + 16 * (i0 + i)) * 128);
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            *reinterpret_cast<uint4 *>(bt + (r0 + 16 * (i0 + i)) * 128) =
                                quantize_f16x8(v[i], nz, rr, qmax_in);
                    }
                }
                fence_proxy_async_smem();  // these stores before the tensor core's reads of b[]
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.bfull[s]));
            }
        }
    } else {
        if constexpr (kTok != kTokF16) regs_inc<144>();
        constexpr int CPW = BN / 2;              // accumulator columns per epilogue warp
        constexpr int PIECE = CPW < 32 ? CPW : 32;
        const int e = warp - kWarpEpi0;
        const int q = warp & 3;
        const int col0 = (e >> 2) * CPW;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t g = 0;
        bool ok = true;
        const int row = q * 32 + lane;  // weight row of the tile
        unsigned long long *flags =
            ws ? reinterpret_cast<unsigned long long *>(ws + (size_t)ws_pairs * 2 * pair_slot_ints()) : nullptr;
        for (int p = 0; p < sch.count && ok; ++p) {
            int u, pk0, pk1;
            sch.piece(p, u, pk0, pk1);
            const int m0 = (u % m_tiles) * BN, n0 = (u / m_tiles) * kBM;
            int32_t tot[CPW];
#pragma unroll
            for (int j = 0; j < CPW; ++j) tot[j] = 0;
            for (int kb0 = pk0; kb0 < pk1; kb0 += kcb, ++g) {
                const int buf = g & 1;
                if (!(ok = mbar_wait(smem_u32(&S.accfull[buf]), (g >> 1) & 1, abort, &g_status))) break;
                tc_fence_after();
                const uint32_t base = tmem + lane_base + kTmemAccCol + buf * BN + col0;
#pragma unroll
                for (int p = 0; p < CPW / PIECE; ++p) {
                    uint32_t v[PIECE];
                    if constexpr (PIECE == 32) tmem_ld32(base + p * 32, v);
                    else if constexpr (PIECE == 16) tmem_ld16(base + p * 16, v);
                    else tmem_ld8(base + p * 8, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int j = 0; j < PIECE; ++j) tot[p * PIECE + j] += __float2int_rn(__uint_as_float(v[j]));
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.accempty[buf]));
            }
            if (!ok) break;
            if (pk1 < nkb) {
                // partial piece: publish the int32 sums for the CTA that ends this tile
                int32_t *slot = ws + (size_t)blockIdx.x * pair_slot_ints();
                if (OT_DCHECK(blockIdx.x < 2u * (unsigned)ws_pairs && col0 + CPW <= 256))
#pragma unroll
                    for (int j = 0; j < CPW; ++j) slot[(size_t)(col0 + j) * 128 + row] = tot[j];
                __threadfence();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.pub));
                // a CTA has at most one partial piece per launch: phase 0 of pub
                if (warp == kWarpEpi0 && lane == 0 && mbar_wait(smem_u32(&S.pub), 0, abort, &g_status)) {
                    __threadfence();
                    atomicExch(flags + blockIdx.x, S.epoch);
                }
                continue;
            }
            if (pk0 > 0) {
                // this CTA ends the tile: add the partial sums of the CTAs that began it
                const int c_lo = sch.first_owner(u);
                for (int c = c_lo; c < (int)blockIdx.x && ok; ++c) {
                    const unsigned long long *f = flags + c;
                    const uint64_t t0 = globaltimer_ns();
                    while (ld_acquire_u64(f) != S.epoch) {
                        if (*abort) { ok = false; break; }
                        if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
                            atomicExch(&g_status, (int)OT_ERR_TIMEOUT);
                            *abort = 1;
                            ok = false;
                            break;
                        }
                    }
                    if (!ok) break;
                    const int32_t *slot = ws + (size_t)c * pair_slot_ints();
#pragma unroll
                    for (int j = 0; j < CPW; ++j) tot[j] += __ldcg(slot + (size_t)(col0 + j) * 128 + row);
                }
                if (!ok) break;
            }
            const int n = n0 + q * 32 + lane;
            if (n < N) {
                if constexpr (kS32) {
                    int32_t *o = reinterpret_cast<int32_t *>(out);
#pragma unroll
                    for (int j = 0; j < CPW; ++j) {
                        const int m = m0 + col0 + j;
                        if (m < M && OT_DCHECK((int64_t)m * N + n < (int64_t)M * N)) o[(int64_t)m * N + n] = tot[j];
                    }
                } else {
                    const float scale = __ldg(sw + n), bias = __ldg(bfold + n);
                    const int32_t zn = kAsym ? __ldg(zc + n) : 0;
                    // chained epilogue: the next layer's z', r' for channel n
                    const float zqn = kQOut ? __ldg(zq + n) : 0.f, rqn = kQOut ? __ldg(rq + n) : 0.f;
                    __half *o = reinterpret_cast<__half *>(out);
#pragma unroll
                    for (int j = 0; j < CPW; ++j) {
                        const int m = m0 + col0 + j;
                        const int mc = m < M ? m : M - 1;
                        // per-token path (Eq. 3): one fp32 product s_m * sw_n
                        const float sc = s_tok ? __fmul_rn(__ldg(s_tok + mc), scale) : scale;
                        // asymmetric weights: sum_k q (qw - zc_n) = acc - zc_n * rowsum_m; the
                        // entry point bounds it below 2^31, so int32 arithmetic (wrapping in between)
                        // gives it exactly
                        const float a = __int2float_rn(kAsym ? (int32_t)((uint32_t)tot[j] -
                                                                          (uint32_t)zn * (uint32_t)__ldg(rowsum + mc))
                                                             : tot[j]);
                        float v = __fmaf_rn(a, sc, bias);
                        if (relu) v = fmaxf(v, 0.f);
                        if constexpr (kQOut) {
                            // the next layer's code round((v - z') * r'), as an fp16 integer
                            const int c = __float2int_rn(__fmul_rn(__fsub_rn(v, zqn), rqn));
                            if (m < M && OT_DCHECK((int64_t)m * ldy + n < (int64_t)(M - 1) * ldy + N))
                                o[(int64_t)m * ldy + n] = __int2half_rn(max(-qmax_out, min(qmax_out, c)));
                        } else {
                            if (m < M && OT_DCHECK((int64_t)m * ldy + n < (int64_t)(M - 1) * ldy + N))
                                o[(int64_t)m * ldy + n] = __float2half_rn(v);
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kWarpAlloc) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (ws && threadIdx.x == 0) {
        unsigned long long *ctl = pair_ctl(ws, ws_pairs);
        if (atomicAdd(ctl + 1, 1ull) == (unsigned long long)gridDim.x - 1) {
            // the last CTA of the launch: hand the epoch to the next launch
            ctl[1] = 0;
            ctl[0] = S.epoch;
        }
    }
}

// ---------------------------------------------------------------------------
// Wide-tile CTA-pair variant: prefill-sized token counts (M > 128, 192-token
// tiles) and 65-128 tokens (128-token tiles; PairCfg below).
//
// Measured on GB300: a cta_group::2 kind::f16 MMA of 256 x N x 16 runs at
// the full tensor rate (4096 MACs per clock per SM, dependent accumulation,
// one commit per 4 MMAs) for every N from 128 to 256, with A in shared
// memory or in TMEM.  TMA copies from L2 cost about 270 ns per copy per SM
// when all SMs stream, whatever their size from 8 to 48 KB (8 KB copies:
// 4.6 TB/s over the GPU; 48 KB copies: 22 TB/s), so the copies must be large:
// one copy per operand brings four 64-wide k-blocks (a 3-D view of the
// row-major array whose outer dimension steps along K).
// So the two CTAs of a cluster run one cta_group::2 MMA of 256 weight rows x
// 192 tokens: per group of four k-blocks each CTA loads its own 128 int8
// weight rows (32 KB, one copy) and half of the token tile (96 rows of fp16
// codes, 48 KB, one copy); B is split along N between the pair and each
// CTA's TMEM receives its 128 rows x 192 tokens of the accumulator (the
// 128-token tile: 64 token rows per CTA, 32 KB copies).
// The converters widen each CTA's int8 weight rows to fp16 and store them in
// TMEM as the MMA's A operand (tcgen05.st), so shared memory carries only
// the TMA ingest, the converters' read of the int8 rows and the tensor
// core's read of B.  TMEM (512 columns) holds two 192-column chunk
// accumulators -- while the MMA fills one, the epilogue converts the other
// (fp32 -> int32 conversions run at a quarter rate and would otherwise stall
// the tensor core at every chunk boundary) -- and four 32-column A stages
// (the 128-token tile: two 128-column accumulators and eight A stages).
// 192-token tiles cover 2048 tokens with 3 % padding.
//   Rank 0 of the pair issues the MMAs.  The converters and epilogue warps
//   of both CTAs signal rank 0's barriers; rank 0's commits arrive on the
//   barriers of both CTAs (multicast): one per k-block frees its A stage,
//   one per group frees the group's B stage.  A converter waits for its own
//   CTA's B stage as well as its weights, so rank 0's wait on the converters
//   of both CTAs covers both halves of B.
//   Warps: 0 TMA producer, 1 MMA issuer, 2 TMEM allocator (warpgroup 0,
//   48 regs); 4-7 and 16-19 converters, taking the even and the odd k-blocks
//   of the CTA's sequence in turn (72 regs: one warp per 32 TMEM lanes could
//   not keep up); 8-15 epilogue (144 regs: PBN / 2 int32 totals).
//   Needs K % 128 == 0 (the 3-D views must not reach past a row's end);
//   other K use linear_kernel.
// ---------------------------------------------------------------------------
constexpr int kGroupKB = 4;                       // k-blocks per TMA copy
// 20 warps: 0 TMA producer, 1 MMA issuer, 2 TMEM allocator, 4-7 and 16-19
// converters (even / odd k-blocks of the CTA's sequence), 8-15 epilogue
constexpr int kPairThreads = 640;
constexpr int kWarpConv1 = 16;
constexpr int kWStages = 2;                       // weight stages: 2 x 128 rows x 128 int8, 128-byte swizzle (32 KB)
constexpr uint32_t kWStageBytes = 2 * kBM * 128;
// Tile width of a CTA pair: PBN tokens (the MMA's N), PBN / 2 token rows per
// CTA; TMEM holds two PBN-column chunk accumulators and (512 - 2 PBN) / 32
// A stages.  Prefill (M > 128) takes 192 or 224 (prefill_tile below): the
// k-loop costs about the same per k-block for any width (measured on GB300:
// ~12 % more at 224, whose MMA is longer and which has two A stages), so the
// fewer token tiles the better -- 4096 tokens in 19 tiles of 224 instead of
// 22 of 192 (OPT-66B fc1 1660 vs 1718 us), 2048 in 11 of 192 rather than 10
// of 224 (9 % padding).  65-128 tokens take 128 (eight A stages).
constexpr int kBStages = 3;                       // token stages: 4 x PBN / 2 rows x 64 fp16, 128-byte swizzle
template <int PBN>
struct PairCfg {
    static constexpr int kBN = PBN;                   // tokens per pair tile (MMA N)
    static constexpr int kHalf = PBN / 2;             // token rows per CTA (B is split along N)
    static constexpr int kACol = 2 * PBN;             // TMEM: accumulators in [0, 2 kBN), then A stages
    static constexpr int kAStg = (512 - kACol) / 32;  // 32-column fp16 A stages (128 rows x 64 k)
    static constexpr uint32_t kBTileBytes = kHalf * 128;
    static constexpr uint32_t kBStageBytes = kGroupKB * kBTileBytes;
    static constexpr int kBStg = PBN > 192 ? 2 : kBStages;  // token stages (224: two, for shared memory)
    static_assert(kAStg >= 2, "A stage of k-block i is freed by the commit of k-block i - kAStg");
    static_assert(kBN % 16 == 0 && kHalf % 16 == 0, "the epilogue drains 16 columns at a time");
    static_assert(kBTileBytes % 1024 == 0, "each k-block of B is a whole number of 1024-byte swizzle atoms");
};
constexpr int kPairBN = 192;  // the prefill tile (also the one pair_max_clusters measures)

// Prefill tile width for M tokens: 224 when its tile count, weighted by its
// ~12 % higher cost per k-block, is below that of 192.
inline int prefill_tile(int64_t M) {
    const int64_t t192 = (M + 191) / 192, t224 = (M + 223) / 224;
    return 28 * t224 < 25 * t192 ? 224 : 192;
}

template <int PBN>
struct alignas(1024) SmemPair {
    using C = PairCfg<PBN>;
    uint8_t b[C::kBStg][C::kBStageBytes];  // this CTA's PBN / 2 token rows of fp16 codes, [k-block][row][64 fp16]
    uint8_t w[kWStages][kWStageBytes];  // this CTA's 128 weight rows of int8 codes, [k-block pair][row][128 int8]
    uint64_t wfull[kWStages];           // own weight copy landed
    uint64_t wempty[kWStages];          // own 4 converter warps read the group's weights
    uint64_t bfull[C::kBStg];           // own token copy landed
    uint64_t bdone[C::kBStg];           // pair MMA of the group done (rank 0 commit, both CTAs)
    uint64_t afull[C::kAStg];           // rank 0 only: both CTAs' converters wrote their A stages (8 warps)
    uint64_t adone[C::kAStg];           // pair MMA of the k-block done (rank 0 commit, both CTAs)
    uint64_t accfull[2];                // pair MMA finished the chunk (rank 0 commit)
    uint64_t accempty[2];               // rank 0 only: both CTAs' epilogues drained the chunk (2 x 8 warps)
    uint64_t pub;                       // stream-K: the 8 epilogue warps stored their partial sums
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    unsigned long long epoch;  // stream-K: this launch's flag value
};

// Groups: a piece's k-blocks [kb0, kb1) are cut at multiples of kGroupKB;
// each group takes one token copy starting at its first k-block and one
// weight copy starting at the even k-block at or below it.
__device__ __forceinline__ bool group_start(int kb, int kb0) { return kb == kb0 || (kb & (kGroupKB - 1)) == 0; }
__device__ __forceinline__ bool group_end(int kb, int kb1) {
    return kb == kb1 - 1 || (kb & (kGroupKB - 1)) == kGroupKB - 1;
}

template <int PBN, bool kS32, bool kAsym, bool kQOut>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
    linear_pair_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_w,
                       const float *__restrict__ sw, const float *__restrict__ bfold, void *__restrict__ out, int M,
                       int N, int K, int ldy, int kcb, int relu, int32_t *__restrict__ ws,
                       const float *__restrict__ s_tok, const int32_t *__restrict__ zc,
                       const int32_t *__restrict__ rowsum, const float *__restrict__ zq,
                       const float *__restrict__ rq, int qmax_out, int group_m) {
    using C = PairCfg<PBN>;
    extern __shared__ uint8_t smem_raw[];
    SmemPair<PBN> &S =
        *reinterpret_cast<SmemPair<PBN> *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = warp_id(), lane = lane_id();
    const uint32_t rank = cluster_ctarank();
    const int cluster = blockIdx.x >> 1, nclusters = gridDim.x >> 1;
    const int m_tiles = (M + C::kBN - 1) / C::kBN;
    const int n_pairs = (N + 2 * kBM - 1) / (2 * kBM);
    const int num_units = m_tiles * n_pairs;
    const int nkb = (K + kBK - 1) / kBK;
    volatile int *abort = &S.abort;
    constexpr uint16_t kBoth = 0x3;
    PairSched sch;
    sch.init(num_units, nkb, nclusters, cluster, ws != nullptr);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kWStages; ++s) {
            mbar_init(smem_u32(&S.wfull[s]), 1);
            mbar_init(smem_u32(&S.wempty[s]), 8);
        }
        for (int s = 0; s < C::kBStg; ++s) {
            mbar_init(smem_u32(&S.bfull[s]), 1);
            mbar_init(smem_u32(&S.bdone[s]), 1);
        }
        for (int s = 0; s < C::kAStg; ++s) {
            mbar_init(smem_u32(&S.afull[s]), 8);
            mbar_init(smem_u32(&S.adone[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&S.accfull[b]), 1);
            mbar_init(smem_u32(&S.accempty[b]), 2 * kNumEpiWarps);
        }
        mbar_init(smem_u32(&S.pub), kNumEpiWarps);
        mbar_init(smem_u32(&S.drain), 1);
        S.abort = 0;
        fence_barrier_init();
        // Launched as a programmatic dependent, the kernel before this one may
        // still be running: prefetch the first weights into L2 (coherent with
        // any write it makes), then wait for it before anything reads the
        // codes or the workspace.
        if (sch.count > 0) {
            int u, pk0, pk1, mt, np;
            sch.piece(0, u, pk0, pk1);
            pair_tile(u, m_tiles, n_pairs, group_m, mt, np);
            tma_prefetch_l2_3d(&tm_w, 0, (np * 2 + (int)rank) * kBM, pk0 >> 1);
        }
        grid_dep_wait();
        S.epoch = ws ? __ldcg(pair_ctl(ws, nclusters)) + 1 : 0;
    }
    if (warp == kWarpTma && lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_w);
    }
    if (warp == kWarpAlloc) {
        tmem_alloc_pair(smem_u32(&S.tmem_base), kTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // barriers of both CTAs exist before either signals the other
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    // the next linear on the stream may launch now (it waits for this one before reading anything this writes)
    grid_dep_launch();

    // registers at launch: 640 threads x 96; after the split 48 / 72 / 144 / 144 / 72 per warpgroup
    if (warp < 4) {
        regs_dec<48>();
        if (warp == kWarpTma) {
            uint32_t gi = 0;
            bool ok = true;
            for (int p = 0; p < sch.count && ok; ++p) {
                int u, pk0, pk1;
                sch.piece(p, u, pk0, pk1);
                int mt, np;
                pair_tile(u, m_tiles, n_pairs, group_m, mt, np);
                const int m0 = mt * C::kBN + (int)rank * C::kHalf;
                const int n0 = (np * 2 + (int)rank) * kBM;
                for (int g0 = pk0; g0 < pk1; g0 = (g0 | (kGroupKB - 1)) + 1, ++gi) {
                    const int ws = gi % kWStages, bs = gi % C::kBStg;
                    // stages last used by group gi - stages: the converters / the pair MMA are done with them
                    if (!(ok = mbar_wait_warp(smem_u32(&S.wempty[ws]), ((gi / kWStages) & 1) ^ 1, abort, &g_status)))
                        break;
                    if (!(ok = mbar_wait_warp(smem_u32(&S.bdone[bs]), ((gi / C::kBStg) & 1) ^ 1, abort, &g_status)))
                        break;
                    if (elect_one()) {
                        mbar_arrive_expect_tx(smem_u32(&S.wfull[ws]), kWStageBytes);
                        tma_load_3d(smem_u32(S.w[ws]), &tm_w, smem_u32(&S.wfull[ws]), 0, n0, g0 >> 1);
                        mbar_arrive_expect_tx(smem_u32(&S.bfull[bs]), C::kBStageBytes);
                        tma_load_3d(smem_u32(S.b[bs]), &tm_q, smem_u32(&S.bfull[bs]), 0, m0, g0);
                    }
                    __syncwarp();
                }
            }
            // teardown: every copy issued must have landed before the CTA exits
            if (lane == 0) {
                for (uint32_t j = gi > (uint32_t)kWStages ? gi - kWStages : 0; j < gi; ++j)
                    wait_teardown(smem_u32(&S.wfull[j % kWStages]), (j / kWStages) & 1);
                for (uint32_t j = gi > (uint32_t)C::kBStg ? gi - C::kBStg : 0; j < gi; ++j)
                    wait_teardown(smem_u32(&S.bfull[j % C::kBStg]), (j / C::kBStg) & 1);
            }
            __syncwarp();
        } else if (warp == kWarpMma && rank == 0) {
            // the whole warp runs the loop and waits; one elected lane issues the MMAs and commits
            const uint32_t idesc = idesc_f16_f32(2 * kBM, C::kBN);
            const uint32_t a_tm = tmem + C::kACol;
            uint32_t it = 0, g = 0, gi = 0, b_base = 0;
            int g0 = 0, bs = 0;
            bool ok = true;
            for (int p = 0; p < sch.count && ok; ++p) {
                int u, pk0, pk1;
                sch.piece(p, u, pk0, pk1);
                for (int kb0 = pk0; kb0 < pk1 && ok; kb0 += kcb, ++g) {
                    const int buf = g & 1;
                    if (!(ok = mbar_wait_warp(smem_u32(&S.accempty[buf]), ((g >> 1) & 1) ^ 1, abort, &g_status)))
                        break;
                    tc_fence_after();
                    const uint32_t d = tmem + buf * C::kBN;
                    const int kb1 = min(pk1, kb0 + kcb);
                    for (int kb = kb0; kb < kb1; ++kb, ++it) {
                        if (group_start(kb, pk0)) {
                            bs = gi % C::kBStg;
                            g0 = kb;
                            b_base = smem_u32(S.b[bs]);
                            ++gi;
                        }
                        const int sa = it % C::kAStg;
                        // both CTAs' converters wrote A stage sa, after their B stage landed
                        if (!(ok = mbar_wait_warp(smem_u32(&S.afull[sa]), (it / C::kAStg) & 1, abort, &g_status)))
                            break;
                        tc_fence_after();
                        const uint64_t bdesc = smem_desc_sw128(b_base + (uint32_t)(kb - g0) * C::kBTileBytes);
                        if (elect_one()) {
#pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk)
                                mma_f16_ts_pair(d, a_tm + sa * 32 + kk * 8, bdesc + (uint64_t)((kk * 32) >> 4), idesc,
                                                (kb != kb0 || kk != 0) ? 1u : 0u);
                            mma_commit_pair_mc(smem_u32(&S.adone[sa]), kBoth);
                            if (group_end(kb, pk1)) mma_commit_pair_mc(smem_u32(&S.bdone[bs]), kBoth);
                        }
                        __syncwarp();
                    }
                    if (ok && elect_one()) mma_commit_pair_mc(smem_u32(&S.accfull[buf]), kBoth);
                    __syncwarp();
                }
            }
            if (elect_one()) {
                mma_commit_pair_mc(smem_u32(&S.drain), 0x1);
                wait_teardown(smem_u32(&S.drain), 0);
            }
            __syncwarp();
        }
    } else if (warp < kWarpEpi0 || warp >= kWarpConv1) {
        regs_dec<72>();
        // converters: warps 4-7 widen the even k-blocks of the CTA's sequence,
        // warps 16-19 the odd ones; both release each weight stage
        const uint32_t set = warp >= kWarpConv1 ? 1u : 0u;
        const int row = (warp & 3) * 32 + lane;  // weight row = TMEM lane
        const uint32_t afull0 = mapa_shared(smem_u32(&S.afull[0]), 0);
        const uint32_t a_tm = tmem + ((uint32_t)((warp & 3) * 32) << 16) + C::kACol;
        uint32_t it = 0, gi = 0;
        int wst = 0, w0 = 0;
        bool gwait = false, ok = true;
        for (int p = 0; p < sch.count && ok; ++p) {
            int u, pk0, pk1;
            sch.piece(p, u, pk0, pk1);
            for (int kb = pk0; kb < pk1; ++kb, ++it) {
                if (group_start(kb, pk0)) {
                    wst = gi % kWStages;
                    w0 = kb & ~1;  // the weight copy starts at this even k-block
                    ++gi;
                    gwait = false;
                }
                const bool last = group_end(kb, pk1);
                if ((it & 1u) != set) {
                    if (last) {
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_u32(&S.wempty[wst]));
                    }
                    continue;
                }
                if (!gwait) {
                    const uint32_t gp = gi - 1;
                    if (!(ok = mbar_wait(smem_u32(&S.wfull[wst]), (gp / kWStages) & 1, abort, &g_status))) break;
                    // the pair MMA reads this CTA's half of B: it must have landed before afull
                    if (!(ok = mbar_wait(smem_u32(&S.bfull[gp % C::kBStg]), (gp / C::kBStg) & 1, abort, &g_status)))
                        break;
                    gwait = true;
                }
                const int sa = it % C::kAStg;
                // this row's 64 bytes of k-block kb: line (kb - w0) / 2 of 128 bytes, 16-byte chunks
                // (kb - w0) % 2 * 4 + c, placed by the 128-byte swizzle at chunk ^ (row % 8)
                const int j = kb - w0;
                const uint8_t *line = S.w[wst] + (j >> 1) * (kBM * 128) + row * 128;
                uint4 raw[4];
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    raw[c] = *reinterpret_cast<const uint4 *>(line + ((((j & 1) * 4 + c) ^ (row & 7)) << 4));
                __syncwarp();
                // the group's last weights are in registers: the stage may be refilled
                if (lane == 0 && last) mbar_arrive(smem_u32(&S.wempty[wst]));
                // the row's 64 fp16 values, two per 32-bit TMEM column, k ascending; widened
                // before waiting for the A stage, so only the TMEM store follows the wait
                uint32_t h[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    i8x4_to_f16x4(raw[c].x, h[8 * c + 0], h[8 * c + 1]);
                    i8x4_to_f16x4(raw[c].y, h[8 * c + 2], h[8 * c + 3]);
                    i8x4_to_f16x4(raw[c].z, h[8 * c + 4], h[8 * c + 5]);
                    i8x4_to_f16x4(raw[c].w, h[8 * c + 6], h[8 * c + 7]);
                }
                // A stage sa was last read by the MMA of k-block it - C::kAStg
                if (it >= (uint32_t)C::kAStg) {
                    const uint32_t prev = it - C::kAStg;
                    if (!(ok = mbar_wait(smem_u32(&S.adone[sa]), (prev / C::kAStg) & 1, abort, &g_status)))
                        break;
                    tc_fence_after();
                }
                tmem_st32(a_tm + sa * 32, h);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(afull0 + (uint32_t)(sa * sizeof(uint64_t)));
            }
        }
    } else {
        regs_inc<144>();
        const int e = warp - kWarpEpi0;
        const int q = warp & 3;
        const int col0 = (e >> 2) * C::kHalf;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const uint32_t accempty0 = mapa_shared(smem_u32(&S.accempty[0]), 0);
        uint32_t g = 0;
        bool ok = true;
        const int row = q * 32 + lane;  // weight row of the CTA's 128
        int32_t *slots = ws;
        unsigned long long *flags =
            ws ? reinterpret_cast<unsigned long long *>(ws + (size_t)nclusters * 2 * pair_slot_ints()) : nullptr;
        for (int p = 0; p < sch.count && ok; ++p) {
            int u, pk0, pk1;
            sch.piece(p, u, pk0, pk1);
            int mt, np;
            pair_tile(u, m_tiles, n_pairs, group_m, mt, np);
            const int m0 = mt * C::kBN;
            const int n0 = (np * 2 + (int)rank) * kBM;
            int32_t tot[C::kHalf];
#pragma unroll
            for (int j = 0; j < C::kHalf; ++j) tot[j] = 0;
            for (int kb0 = pk0; kb0 < pk1; kb0 += kcb, ++g) {
                const int buf = g & 1;
                if (!(ok = mbar_wait(smem_u32(&S.accfull[buf]), (g >> 1) & 1, abort, &g_status))) break;
                tc_fence_after();
                const uint32_t base = tmem + lane_base + buf * C::kBN + col0;
#pragma unroll
                for (int p = 0; p < C::kHalf / 16; ++p) {
                    uint32_t v[16];
                    tmem_ld16(base + p * 16, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int j = 0; j < 16; ++j) tot[p * 16 + j] += __float2int_rn(__uint_as_float(v[j]));
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(accempty0 + (uint32_t)(buf * sizeof(uint64_t)));
            }
            if (!ok) break;
            if (pk1 < nkb) {
                // partial piece: publish the int32 sums for the pair that ends this tile
                int32_t *slot = slots + ((size_t)cluster * 2 + rank) * pair_slot_ints();
                if (OT_DCHECK(cluster < nclusters && col0 + C::kHalf <= 256))
#pragma unroll
                    for (int j = 0; j < C::kHalf; ++j) slot[(size_t)(col0 + j) * 128 + row] = tot[j];
                __threadfence();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&S.pub));
                // a pair has at most one partial piece per launch: phase 0 of pub
                if (warp == kWarpEpi0 && lane == 0 && mbar_wait(smem_u32(&S.pub), 0, abort, &g_status)) {
                    __threadfence();
                    atomicExch(flags + (size_t)cluster * 2 + rank, S.epoch);
                }
                continue;
            }
            if (pk0 > 0) {
                // this pair ends the tile: add the partial sums of the pairs that began it
                const int c_lo = sch.first_owner(u);
                for (int c = c_lo; c < cluster && ok; ++c) {
                    const unsigned long long *f = flags + (size_t)c * 2 + rank;
                    const uint64_t t0 = globaltimer_ns();
                    while (ld_acquire_u64(f) != S.epoch) {
                        if (*abort) { ok = false; break; }
                        if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
                            atomicExch(&g_status, (int)OT_ERR_TIMEOUT);
                            *abort = 1;
                            ok = false;
                            break;
                        }
                    }
                    if (!ok) break;
                    const int32_t *slot = slots + ((size_t)c * 2 + rank) * pair_slot_ints();
#pragma unroll
                    for (int j = 0; j < C::kHalf; ++j) tot[j] += __ldcg(slot + (size_t)(col0 + j) * 128 + row);
                }
                if (!ok) break;
            }
            const int n = n0 + q * 32 + lane;
            if (n < N) {
                if constexpr (kS32) {
                    int32_t *o = reinterpret_cast<int32_t *>(out);
#pragma unroll
                    for (int j = 0; j < C::kHalf; ++j) {
                        const int m = m0 + col0 + j;
                        if (m < M && OT_DCHECK((int64_t)m * N + n < (int64_t)M * N)) o[(int64_t)m * N + n] = tot[j];
                    }
                } else {
                    const float scale = __ldg(sw + n), bias = __ldg(bfold + n);
                    const int32_t zn = kAsym ? __ldg(zc + n) : 0;
                    // chained epilogue: the next layer's z', r' for channel n
                    const float zqn = kQOut ? __ldg(zq + n) : 0.f, rqn = kQOut ? __ldg(rq + n) : 0.f;
                    __half *o = reinterpret_cast<__half *>(out);
#pragma unroll
                    for (int j = 0; j < C::kHalf; ++j) {
                        const int m = m0 + col0 + j;
                        const int mc = m < M ? m : M - 1;
                        // per-token path (Eq. 3): one fp32 product s_m * sw_n
                        const float sc = s_tok ? __fmul_rn(__ldg(s_tok + mc), scale) : scale;
                        // asymmetric weights: sum_k q (qw - zc_n) = acc - zc_n * rowsum_m; the
                        // entry point bounds it below 2^31, so int32 arithmetic (wrapping in between)
                        // gives it exactly
                        const float a = __int2float_rn(kAsym ? (int32_t)((uint32_t)tot[j] -
                                                                          (uint32_t)zn * (uint32_t)__ldg(rowsum + mc))
                                                             : tot[j]);
                        float v = __fmaf_rn(a, sc, bias);
                        if (relu) v = fmaxf(v, 0.f);
                        if constexpr (kQOut) {
                            // the next layer's code round((v - z') * r'), as an fp16 integer
                            const int c = __float2int_rn(__fmul_rn(__fsub_rn(v, zqn), rqn));
                            if (m < M && OT_DCHECK((int64_t)m * ldy + n < (int64_t)(M - 1) * ldy + N))
                                o[(int64_t)m * ldy + n] = __int2half_rn(max(-qmax_out, min(qmax_out, c)));
                        } else {
                            if (m < M && OT_DCHECK((int64_t)m * ldy + n < (int64_t)(M - 1) * ldy + N))
                                o[(int64_t)m * ldy + n] = __float2half_rn(v);
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync();  // no CTA of the pair touches the other's memory or barriers after this
    if (warp == kWarpAlloc) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, kTmemCols);
    }
    if (ws && threadIdx.x == 0) {
        unsigned long long *ctl = pair_ctl(ws, nclusters);
        if (atomicAdd(ctl + 1, 1ull) == (unsigned long long)gridDim.x - 1) {
            // the last CTA of the launch: hand the epoch to the next launch
            ctl[1] = 0;
            ctl[0] = S.epoch;
        }
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
constexpr int64_t kStreamKMinSaving = 32;  // k-blocks per worker

// Whether stream-K pays for `units` tiles of `nkb` k-blocks over `workers`:
// when it shortens the busiest worker's share by at least kStreamKMinSaving
// k-blocks, or, when there are fewer tiles than workers (some would idle for
// the whole launch), by at least 1 / idle_div of a tile (idle_div 0: never).
// Measured on GB300 at 32-192 tokens (OPT-6.7B QKV / fc1, OPT-13B QKV, whose
// tiles are 63-80 % of the workers): the CTA kernel gains once the share is a
// fifth shorter (37 %: 15 % faster, 21 %: 5 %; 16 %: 1.5 % slower), the
// 128-token pair tile once it is a third shorter (37 %: 6.5 % faster; 21 % and
// 16 %: 2 and 9 % slower), the 192-token pair tile at none of these.
inline bool streamk_pays(int64_t units, int64_t nkb, int64_t workers, int64_t idle_div) {
    const int64_t whole = (units + workers - 1) / workers * nkb;
    const int64_t shared = (units * nkb + workers - 1) / workers;
    const int64_t saving = whole - shared;
    return saving >= kStreamKMinSaving || (idle_div > 0 && units < workers && idle_div * saving >= whole);
}

size_t pair_workspace_bytes(int clusters) {
    return (size_t)clusters * 2 * pair_slot_ints() * sizeof(int32_t) + (size_t)clusters * 2 * sizeof(uint64_t) +
           2 * sizeof(uint64_t);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

bool make_tmap_2d(CUtensorMap *tm, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
                  uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle swz) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(tm, dt, 2, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// 3-D view {inner, rows, outer} of a row-major array with `row_bytes` per
// row: element (i, r, o) sits at base + r row_bytes + o outer_bytes + i * size.
// With outer_bytes equal to the inner span the view covers each row once, as
// consecutive slices along it.
bool make_tmap_3d(CUtensorMap *tm, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
                  uint64_t outer, uint64_t row_bytes, uint64_t outer_bytes, uint32_t box_inner, uint32_t box_rows,
                  uint32_t box_outer, CUtensorMapSwizzle swz) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {inner, rows, outer};
    cuuint64_t strides[2] = {row_bytes, outer_bytes};
    cuuint32_t box[3] = {box_inner, box_rows, box_outer};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(tm, dt, 3, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int pair_max_clusters();

template <int BN, bool kS32, bool kAsym, bool kQOut, int kTok>
cudaError_t run_linear(const LinearArgs &a, int kcb, cudaStream_t st) {
    // token tiles: BN rows x 64 channels of fp16 codes or fp16 activations
    // (128-byte swizzle, the MMA's layout) or of int8 codes (unswizzled, widened
    // by the token warps); weights: 128 rows x 64 int8 (64-byte swizzle)
    CUtensorMap tm_q, tm_w;
    const bool qmap = kTok == kTokI8
                          ? make_tmap_2d(&tm_q, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.q, (uint64_t)a.K, (uint64_t)a.M,
                                         (uint64_t)a.K, kBK, BN, CU_TENSOR_MAP_SWIZZLE_NONE)
                          : make_tmap_2d(&tm_q, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a.q, (uint64_t)a.K, (uint64_t)a.M,
                                         (uint64_t)(kTok == kTokX ? a.ldx : a.K) * 2, kBK, BN,
                                         CU_TENSOR_MAP_SWIZZLE_128B);
    if (!qmap || !make_tmap_2d(&tm_w, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.qw, (uint64_t)a.K, (uint64_t)a.N,
                               (uint64_t)a.K, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_64B))
        return cudaErrorInvalidValue;
    // at least 120 KB so two CTAs never share an SM (each takes all 512 TMEM columns)
    using SmemT = Smem<BN, kTok>;
    const size_t smem = sizeof(SmemT) + 1024 > 120 * 1024 ? sizeof(SmemT) + 1024 : 120 * 1024;
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(linear_kernel<BN, kS32, kAsym, kQOut, kTok>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (attr_err != cudaSuccess) return attr_err;
    const int64_t tiles = ((a.M + BN - 1) / BN) * ((a.N + kBM - 1) / kBM);
    const int64_t nkb = (a.K + kBK - 1) / kBK;
    // Stream-K over CTAs, in the prefill kernel's workspace layout (a slot and
    // a flag per CTA; one CTA per SM, at most 2 x pair_max_clusters of them),
    // when streamk_pays (e.g. OPT-13B fc2 at 64 tokens: 40 tiles of 320
    // k-blocks; OPT-6.7B QKV: 96 tiles of 64 k-blocks on 152 CTAs).
    const int pairs = pair_max_clusters();
    const int workers = num_sms() < 2 * pairs ? num_sms() : 2 * pairs;
    const bool streamk = a.workspace != nullptr && a.workspace_bytes >= pair_workspace_bytes(pairs) &&
                         streamk_pays(tiles, nkb, workers, 5) && tiles * nkb < ((int64_t)1 << 30);
    const int grid = streamk ? workers : (int)(tiles < num_sms() ? tiles : num_sms());
    int32_t *ws = streamk ? reinterpret_cast<int32_t *>(a.workspace) : nullptr;
    return launch_kernel(linear_kernel<BN, kS32, kAsym, kQOut, kTok>, dim3(grid), dim3(lin_threads<kTok>()), smem,
                         st, a.pdl, tm_q, tm_w, a.sw, a.bfold, a.out, (int)a.M, (int)a.N, (int)a.K, (int)a.ldy, kcb,
                         a.relu, a.s_tok, a.zc, a.rowsum, a.zq, a.rq, a.qmax_out, ws, pairs, a.xz, a.xr, a.qmax_in);
}

// Clusters of the pair kernel that fit on the device at once (one per two SMs).
int pair_max_clusters() {
    static int dev_cached = -1, value = 0;
    static std::mutex mu;
    int dev = 0;
    cudaGetDevice(&dev);
    std::lock_guard<std::mutex> lock(mu);
    if (dev_cached == dev) return value;
    const size_t smem = sizeof(SmemPair<kPairBN>) + 1024;
    int n = 0;
    if (cudaFuncSetAttribute(linear_pair_kernel<kPairBN, false, false, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) ==
        cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * 256);
        cfg.blockDim = dim3(kPairThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = 2;
        attr.val.clusterDim.y = 1;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, linear_pair_kernel<kPairBN, false, false, false>, &cfg) != cudaSuccess)
            n = 0;
    }
    cudaGetLastError();
    if (n <= 0) n = num_sms() / 2;
    dev_cached = dev;
    value = n;
    return n;
}

// Token tiles per group of the pair kernel's tile order (pair_tile), from an
// estimate of the DRAM bytes each order reads.  Two estimates, the smaller
// taken:
//  - L2 keeps a group's codes while the weight tiles stream past them: the
//    codes are read once, the weights once per group (when G token tiles of
//    codes fit beside the stream).  Measured on GB300: OPT-66B fc1 (4096
//    tokens, K = 9216; 75 MB of codes) read 3.3 GB per launch in the plain
//    order, 1.17 GB with 11 token tiles per group, against 415 MB of operands.
//  - otherwise the clusters of one round (a tile each, moving along k at
//    about the same pace) share what they read at about the same time, so a
//    round reads the distinct token tiles and weight tiles it touches.  With
//    K = 36864 (OPT-66B fc2) a tile's operands alone are 24 MB: 7 token
//    tiles per group read 3.0 GB per launch against 4.0 GB in the plain order
//    (and ran 2 % faster).
int pair_group_m(int64_t M, int64_t N, int64_t K, int clusters, int pbn) {
    constexpr double kL2Keep = 48.0 * (1 << 20);  // codes a group may keep in L2 beside the weight stream
    const int64_t m_tiles = (M + pbn - 1) / pbn;
    const int64_t n_pairs = (N + 2 * kBM - 1) / (2 * kBM);
    const int64_t cl = clusters > 0 ? clusters : 1;
    const double tile_codes = (double)pbn * (double)K * 2.0, tile_weights = 2.0 * kBM * (double)K;
    const double codes = tile_codes * (double)m_tiles, weights = (double)N * (double)K;
    const double rounds = std::max(1.0, (double)(m_tiles * n_pairs) / (double)cl);
    auto per_rounds = [&](int64_t g) {
        int64_t toks, prs;
        if (cl <= g * n_pairs) {
            toks = std::min(g, cl);
            prs = (cl + g - 1) / g;
        } else {
            toks = std::min(m_tiles, (cl + n_pairs - 1) / n_pairs);
            prs = n_pairs;
        }
        return rounds * ((double)toks * tile_codes + (double)prs * tile_weights);
    };
    const double plain = codes <= kL2Keep ? std::min(codes + weights, per_rounds(m_tiles)) : per_rounds(m_tiles);
    int64_t best_g = m_tiles;
    double best = plain;
    for (int64_t g = 1; g < m_tiles; ++g) {
        double t = per_rounds(g);
        if ((double)g * tile_codes <= kL2Keep) t = std::min(t, codes + (double)((m_tiles + g - 1) / g) * weights);
        if (t < best) {
            best = t;
            best_g = g;
        }
    }
    return best < 0.8 * plain ? (int)best_g : (int)m_tiles;
}

template <int PBN, bool kS32, bool kAsym, bool kQOut>
cudaError_t run_linear_pair(const LinearArgs &a, int kcb, cudaStream_t st) {
    using C = PairCfg<PBN>;
    // codes as {64 fp16, M rows, K / 64 k-blocks}: a box of 96 rows x 4 k-blocks;
    // weights as {128 int8, N rows, K / 128 k-block pairs}: a box of 128 rows x 2 pairs.
    // Each inner span is a whole slice of the row (K % 128 == 0), so no copy
    // reaches past a row; rows past M or N and k-blocks past K are zero-filled.
    CUtensorMap tm_q, tm_w;
    if (!make_tmap_3d(&tm_q, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a.q, kBK, (uint64_t)a.M, (uint64_t)a.K / kBK,
                      (uint64_t)a.K * 2, kBK * 2, kBK, C::kHalf, kGroupKB, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_tmap_3d(&tm_w, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.qw, 128, (uint64_t)a.N, (uint64_t)a.K / 128,
                      (uint64_t)a.K, 128, 128, kBM, kGroupKB / 2, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    const size_t smem = sizeof(SmemPair<PBN>) + 1024;
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(linear_pair_kernel<PBN, kS32, kAsym, kQOut>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (attr_err != cudaSuccess) return attr_err;
    const int max_clusters = pair_max_clusters();
    const int64_t units = ((a.M + C::kBN - 1) / C::kBN) * ((a.N + 2 * kBM - 1) / (2 * kBM));
    const int64_t nkb = (a.K + kBK - 1) / kBK;
    // Stream-K shortens the busiest pair's work from ceil(units / pairs) whole
    // tiles to an equal share of k-blocks, at the cost of a partial-sum
    // exchange per split tile.  Measured on GB300 it pays off once it saves
    // about 32 k-blocks per pair (OPT-6.7B QKV and fc2 at 2048 tokens: 7-11 %
    // faster; out and fc1, which save ~20, are 1-2 % slower); see streamk_pays.
    const bool streamk = a.workspace != nullptr && a.workspace_bytes >= pair_workspace_bytes(max_clusters) &&
                         streamk_pays(units, nkb, max_clusters, PBN == 128 ? 3 : 0) &&
                         units * nkb < ((int64_t)1 << 30);
    const int clusters = streamk ? max_clusters : (int)(units < max_clusters ? units : max_clusters);
    int32_t *ws = streamk ? reinterpret_cast<int32_t *>(a.workspace) : nullptr;
    const int group_m = pair_group_m(a.M, a.N, a.K, clusters, C::kBN);
    return launch_kernel(linear_pair_kernel<PBN, kS32, kAsym, kQOut>, dim3(2 * clusters), dim3(kPairThreads), smem, st,
                         a.pdl, tm_q, tm_w, a.sw, a.bfold, a.out, (int)a.M, (int)a.N, (int)a.K, (int)a.ldy, kcb, a.relu,
                         ws, a.s_tok, a.zc, a.rowsum, a.zq, a.rq, a.qmax_out, group_m);
}

// M <= 16 goes to the decode kernel (gemv.cu) before this dispatch.
template <bool kS32, bool kAsym, bool kQOut>
cudaError_t dispatch_bn(const LinearArgs &a, int kcb, cudaStream_t st) {
    // Measured on GB300 (OPT-13B QKV / fc2): the 128-token pair tile is 2-3 % faster than linear_kernel at
    // 65-128 tokens (QKV 28.2 vs 28.9 us, fc2 36.3 vs 37.2 at 128) and 6-12 % slower at 17-64
    if (a.K % 128 == 0 && a.M > 128)
        return prefill_tile(a.M) == 224 ? run_linear_pair<224, kS32, kAsym, kQOut>(a, kcb, st)
                                        : run_linear_pair<kPairBN, kS32, kAsym, kQOut>(a, kcb, st);
    if (a.K % 128 == 0 && a.M > 64) return run_linear_pair<128, kS32, kAsym, kQOut>(a, kcb, st);
    if (a.M <= 64) return run_linear<64, kS32, kAsym, kQOut, kTokF16>(a, kcb, st);
    return run_linear<128, kS32, kAsym, kQOut, kTokF16>(a, kcb, st);
}

// int8 codes (any M > 16) and fp16 activations quantized in the kernel
// (16 < M <= 128) go to linear_kernel with its token warps.
template <int kTok>
cudaError_t dispatch_tok(const LinearArgs &a, int kcb, cudaStream_t st) {
    if (a.out_s32)
        return a.M <= 64 ? run_linear<64, true, false, false, kTok>(a, kcb, st)
                         : run_linear<128, true, false, false, kTok>(a, kcb, st);
    return a.M <= 64 ? run_linear<64, false, false, false, kTok>(a, kcb, st)
                     : run_linear<128, false, false, false, kTok>(a, kcb, st);
}

}  // namespace


bool tensor_map_2d(CUtensorMap *tm, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
                   uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle swz) {
    return make_tmap_2d(tm, dt, base, inner, rows, row_bytes, box_inner, box_rows, swz);
}

// Token counts up to this go to the mma.sync weight-streaming kernel (gemv.cu)
// (measured crossover on GB300: OPT-13B QKV at 17-32 tokens 27.0-27.6 us in
// linear_kernel against 27.8-32.0 us in gemv.cu; fc2 33.4-33.6 against 35.0-41.6).
constexpr int64_t kGemvMaxTokens = 16;

// Largest number of 64-wide k-blocks whose fp32 partial sums stay exact:
// kcb * 64 * qmax_a * qmax_w <= 2^24.
int exact_chunk_kblocks(int bits_a, int bits_w, bool asym_w) {
    // asymmetric weight codes are stored as u - 2^(b-1): |qw| <= 2^(b-1)
    const int64_t qa = (1 << (bits_a - 1)) - 1, qw = (1 << (bits_w - 1)) - (asym_w ? 0 : 1);
    int64_t kc = ((int64_t)1 << 24) / (qa * qw);
    kc /= kBK;
    return kc < 1 ? 1 : (int)kc;
}

// Workspace layout: the stream-K region of the prefill kernel, then the
// split-tile region of the decode kernel.
size_t linear_workspace_bytes() { return pair_workspace_bytes(pair_max_clusters()) + gemv_workspace_bytes(); }

int *device_status_word() {
    static std::mutex mu;
    static int *addr[64] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
        addr[dev] = static_cast<int *>(p);
    }
    return addr[dev];
}

// Scratch of ot_linear_noalloc: the stream-K workspace lives in this
// file-scope device array, so that entry point never allocates.  Every GPU
// that loads the library holds it until the process exits.  24 MiB covers
// the prefill and decode partial-sum slots and flags of devices with up to
// 170 SMs (a 152-SM GB300 needs about 22.4 MB).
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch on the current device.  In host code
// the array's name is only a stand-in, so the address comes from
// cudaGetSymbolAddress, once per device, with that device current; the first
// use on a device also zero-fills the array (the stream-K flags and epoch
// counters start at zero; the kernels keep them consistent after that) and
// waits for the fill on `st`, so a call from another thread or stream that
// finds the address cached never runs ahead of the fill.
cudaError_t noalloc_scratch(void **ptr, cudaStream_t st) {
    static std::mutex mu;
    static void *addr[64] = {nullptr};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        e = cudaMemsetAsync(p, 0, kNoAllocScratchBytes, st);
        if (e != cudaSuccess) return e;
        e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *ptr = addr[dev];
    return cudaSuccess;
}

cudaError_t launch_linear(const LinearArgs &args, cudaStream_t st) {
    if (args.M == 0 || args.N == 0) return cudaSuccess;
    // Every linear launches as a programmatic dependent of the kernel before it
    // on the stream, and lets the next one launch once its own set-up is done:
    // consecutive linears overlap one's tail with the next one's launch, set-up
    // and first weight fetches (each kernel reads codes, outputs and workspace
    // only after the one before it has ended).
    LinearArgs a = args;
    a.pdl = true;
    const int nkb = (int)((a.K + kBK - 1) / kBK);
    int kcb = exact_chunk_kblocks(a.bits_a, a.bits_w, a.zc != nullptr);
    if (kcb > nkb) kcb = nkb;
    if (a.M <= kGemvMaxTokens) {
        LinearArgs d = a;
        const size_t off = pair_workspace_bytes(pair_max_clusters());
        const bool room = a.workspace != nullptr && a.workspace_bytes >= off + gemv_workspace_bytes();
        d.workspace = room ? static_cast<unsigned char *>(a.workspace) + off : nullptr;
        d.workspace_bytes = room ? a.workspace_bytes - off : 0;
        return launch_linear_gemv(d, kcb, st);
    }
    if (a.q_fmt == kCodesI8) return dispatch_tok<kTokI8>(a, kcb, st);
    if (a.q_fmt == kActF16) return dispatch_tok<kTokX>(a, kcb, st);
    if (a.out_s32) return dispatch_bn<true, false, false>(a, kcb, st);
    if (a.zq) return dispatch_bn<false, false, true>(a, kcb, st);
    return a.zc ? dispatch_bn<false, true, false>(a, kcb, st) : dispatch_bn<false, false, false>(a, kcb, st);
}

}  // namespace ot

namespace ot {

namespace {
// One thread waits, with the given limit, on an mbarrier that nothing
// arrives on; the expiry takes the same path as the GEMM's bounded waits
// (OT_ERR_TIMEOUT in the device status word) and the kernel returns.
__global__ void wait_timeout_kernel(uint64_t limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(smem_u32(&bar), 1);
    fence_barrier_init();
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(smem_u32(&bar), 0)) {
        if (globaltimer_ns() - t0 > limit_ns) {
            atomicExch(&g_status, (int)OT_ERR_TIMEOUT);
            return;
        }
    }
}
}  // namespace

cudaError_t launch_wait_timeout(int64_t limit_ns, cudaStream_t st) {
    wait_timeout_kernel<<<1, 32, 0, st>>>((uint64_t)limit_ns);
    return cudaGetLastError();
}

cudaError_t read_clear_status(int *value, cudaStream_t st) {
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return e;
    int v = 0;
    e = cudaMemcpyFromSymbol(&v, g_status, sizeof(int));
    if (e != cudaSuccess) return e;
    const int zero = 0;
    e = cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
    *value = v;
    return e;
}

}  // namespace ot
