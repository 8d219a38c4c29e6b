// ot_kernels.h -- host-side launchers of the sm_103a kernels (internal to the
// library; the public boundary is include/outliertune.h).  Every launcher
// assumes its arguments were validated by the C-ABI layer in api.cu and
// returns the launch error of its kernel(s).
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace ot {

cudaError_t launch_calibrate(const void *x, int64_t T, int64_t K, int64_t ldx, float *mn, float *mx, int reset,
                             cudaStream_t st);
cudaError_t launch_params(const float *mn, const float *mx, int64_t K, int bits, int symmetrize, float *z,
                          float *s, float *r, cudaStream_t st);
cudaError_t launch_fold(const void *w, const void *b, int64_t N, int64_t K, const float *z, const float *s,
                        int bits_w, int8_t *qw, float *sw, float *bfold, cudaStream_t st);
// rowsum (optional, int32 [M]): sum_k q[m,k], for the asymmetric-weight epilogue
cudaError_t launch_quantize(const void *x, int64_t M, int64_t K, int64_t ldx, const float *z, const float *r,
                            int bits, void *q, int fmt, cudaStream_t st, int32_t *rowsum = nullptr);
cudaError_t launch_quantize_tokens(const void *x, int64_t M, int64_t K, int64_t ldx, int bits, void *q, int fmt,
                                   float *s_tok, cudaStream_t st);
// token-wise clipping calibration: per-channel order statistics (clip.cu)
cudaError_t launch_calibrate_clipped(const void *x, int64_t T, int64_t K, int64_t ldx, double alpha, float *lo,
                                     float *hi, cudaStream_t st);
// LayerNorm fused with the symmetrization and quantization (layernorm.cu)
cudaError_t launch_fold_layernorm(const void *gamma, const void *beta, const float *z, const float *r, int64_t K,
                                  float *gamma_r, float *beta_r, cudaStream_t st);
cudaError_t launch_layernorm_quantize(const void *h, int64_t M, int64_t K, int64_t ldh, const float *gamma_r,
                                      const float *beta_r, float eps, int bits, void *q, int fmt,
                                      int32_t *rowsum, cudaStream_t st);
// asymmetric per-output-channel codes of W_s (zero points zc) and b'
cudaError_t launch_fold_asym(const void *w, const void *b, int64_t N, int64_t K, const float *z, const float *s,
                             int bits_w, int8_t *qw, float *sw, int32_t *zc, float *bfold, cudaStream_t st);
// per-output-channel weight codes without activation scales (s = 1)
cudaError_t launch_quantize_weights(const void *w, int64_t N, int64_t K, int bits_w, int8_t *qw, float *sw,
                                    cudaStream_t st);

struct LinearArgs {
    const void *q;        // fp16 codes [M, K]
    const int8_t *qw;     // int8 codes [N, K]
    const float *sw;      // [N] (fp16 output only)
    const float *bfold;   // [N] (fp16 output only)
    void *out;            // fp16 y [M, ldy] or int32 acc [M, N]
    int64_t M, N, K, ldy;
    int bits_a, bits_w, relu;
    bool out_s32;
    void *workspace;          // stream-K partial sums (zero-filled before first use) or null
    size_t workspace_bytes;
    const float *s_tok;       // per-token path: token scales [M] (y uses s_tok[m] * sw[n]); null otherwise
    const int32_t *zc;        // asymmetric weights: zero points [N] (stored codes' scale), or null
    const int32_t *rowsum;    // with zc: sum_k q[m,k] [M]
    const float *zq, *rq;     // chained epilogue: the next layer's z', r' [N] (out then holds fp16 codes), or null
    int qmax_out;             // with zq: the next layer's qmax
    bool pdl;                 // (set by launch_linear) launched as a programmatic dependent of the kernel
                              // before it on the stream: the kernel reads codes, outputs and workspace only
                              // after that kernel ends, and may prefetch weights into L2 before
    bool weights_early = false;  // that kernel is this call's own quantize kernel (ot_linear_fused), which
                                 // releases its dependents only after every earlier kernel (any writer of
                                 // the weights) has completed: weights may be loaded before it ends
    int q_fmt = 0;            // kCodesF16: q holds fp16 codes; kCodesI8: int8 codes; kActF16: fp16
                              // activations [M, ldx] that the kernel quantizes with xz, xr, qmax_in
    const float *xz = nullptr, *xr = nullptr;  // kActF16: z, r [K]
    int64_t ldx = 0;          // kActF16: row stride of q
    int qmax_in = 0;          // kActF16: qmax of the codes
};
constexpr int kCodesF16 = 0, kCodesI8 = 1, kActF16 = 2;
// Largest token count for which the linear's token producer can quantize X
// itself (decode kernel and linear_kernel); above it only the prefill kernel,
// reading codes written by the quantize kernel, runs.
constexpr int64_t kFusedInKernelMaxTokens = 128;
// Workspace bytes that enable stream-K scheduling of the prefill kernel on this device.
size_t linear_workspace_bytes();
// Fixed scratch of ot_linear_noalloc (a static device array in gemm.cu).
constexpr size_t kNoAllocScratchBytes = (size_t)24 << 20;
cudaError_t noalloc_scratch(void **ptr, cudaStream_t st);
cudaError_t launch_linear(const LinearArgs &a, cudaStream_t st);
// decode-sized token counts (M <= 32); kcb as in launch_linear; a.workspace is
// the decode region of the caller's workspace (or null)
cudaError_t launch_linear_gemv(const LinearArgs &a, int kcb, cudaStream_t st);
// bytes of the decode region (split-tile partial sums and counters)
size_t gemv_workspace_bytes();
// device address of the status word that bounded waits write on timeout
int *device_status_word();
// 2-D tiled tensor map of a row-major [rows, inner] array (false if the
// driver's encoder is missing or rejects the arguments)
bool tensor_map_2d(CUtensorMap *tm, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
                   uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle swz);

int num_sms();
#ifdef OT_DEBUG
// first failed index check (source line) of each file's kernels since the last read
cudaError_t dbg_read_clear_gemm(unsigned *line);
cudaError_t dbg_read_clear_gemv(unsigned *line);
cudaError_t dbg_read_clear_quant(unsigned *line);
cudaError_t dbg_read_clear_fold(unsigned *line);
#endif
int exact_chunk_kblocks(int bits_a, int bits_w, bool asym_w);
cudaError_t read_clear_status(int *value, cudaStream_t st);
cudaError_t launch_wait_timeout(int64_t limit_ns, cudaStream_t st);

}  // namespace ot
