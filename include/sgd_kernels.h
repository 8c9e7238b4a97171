/*
 * sgd_kernels.h — kernel-level entry points of libsgd, one per hot-path kernel of
 * the scheduled denoiser step.  They exist so that every kernel can be checked
 * against the CPU oracle on its own; sgd_step launches the same kernels with the
 * same launch configurations.
 *
 * Paper passages (Algorithm 2, "Jagged-Stream Execution"):
 *   - an active unit computes Delta_{l,s} = F_l(h_{l-1,s}; c_s), refreshes its cache
 *     and sets h_{l,s} = h_{l-1,s} + Delta   -> sgd_kernel_gemm with SGD_EPI_DELTA
 *     (the branch's last projection, its epilogue stores the cache and adds to h);
 *   - the branch body F_l (norm, projections, attention, MLP activation)
 *                                          -> sgd_kernel_norm, sgd_kernel_gemm,
 *                                             sgd_kernel_attention;
 *   - a frozen unit reads its cached Delta_{l, r_l(s)} and adds it to the current
 *     residual stream                        -> sgd_kernel_frozen_run (one pass over h
 *     for a run of consecutive frozen units).
 *
 * All pointers are device pointers; all calls are asynchronous on `stream`
 * (a cudaStream_t) and return an sgd_status (sgd.h).  Arguments are validated on
 * the host (SGD_ERR_ARG / SGD_ERR_SHAPE); nothing is launched on a validation error.
 */
#ifndef SGD_KERNELS_H
#define SGD_KERNELS_H

#include <stdint.h>

#ifndef SGD_API
#if defined(__GNUC__)
#define SGD_API __attribute__((visibility("default")))
#else
#define SGD_API
#endif
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Epilogue applied to the fp32 accumulator tile of C = A B^T. */
/* acc = alpha * (A B^T), fp32.  fp16 outputs saturate at +-65504. */
typedef enum {
  SGD_EPI_F16 = 0,    /* out fp16 [M, N] = acc                                          */
  SGD_EPI_F32 = 1,    /* out fp32 [M, N] = acc                                          */
  SGD_EPI_DELTA = 2,  /* Delta = gate * acc; h fp32 [M, N] += Delta; cache fp16 = Delta   */
  SGD_EPI_GATED = 3,  /* B has 2f rows; out fp16 [M, f] = act(acc[:, :f], acc[:, f:])   */
  SGD_EPI_GELU = 4,   /* out fp16 [M, N] = gelu(acc)                                    */
  SGD_EPI_ROPE = 5    /* out fp16 [M, N] = acc with rotate-half RoPE on columns < rope_cols */
} sgd_epilogue_kind;

typedef struct {
  int kind;                      /* sgd_epilogue_kind                                        */
  float alpha;                   /* accumulator scale (0 is read as 1)                        */
  void* out; int ldo;            /* output (elements); unused by SGD_EPI_DELTA               */
  float* h; int ldh;             /* DELTA: fp32 residual updated in place                   */
  void* cache; int ld_cache;     /* DELTA: optional fp16 copy of Delta (NULL: not stored)    */
  const float* gate;             /* DELTA: optional fp32 gate [B, ld_gate], row r uses sample r / rows_per_batch */
  int ld_gate, rows_per_batch;
  int act;                       /* GATED: 0 = silu(a) * b (SwiGLU), 1 = a * gelu_erf(b) (GEGLU);
                                    GELU: 0 = tanh form, 1 = erf form                           */
  const float* rope_cos;         /* ROPE: fp32 [rope_tokens, d_head / 2] tables, row = token % rope_tokens */
  const float* rope_sin;
  int rope_tokens, d_head, rope_cols;
  /* Pre-norm folded into the GEMM (Algorithm 2, an active branch's Norm before its first
   * projection): A holds the un-normalised rows x (fp16), B = W diag(g) (the norm gain
   * folded into the weight), and before its epilogue each accumulator value of row r, B
   * row j becomes
   *   SGD_FNORM_RMS (1): rstd_r acc,  rstd_r = rsqrt(sum_p sq[p][r] / K + norm_eps);
   *   SGD_FNORM_LN  (2): rstd_r (acc - mean_r colsum[j]) + colbias[j], with mean_r =
   *                      sum_p s[p][r] / K and rstd_r = rsqrt(sum_p sq[p][r] / K - mean_r^2 + eps),
   * where sq[p][r] = rstat[p * stat_ld + r] and s[p][r] = rstat[(64 + p) * stat_ld + r] are
   * the partial row sums of x^2 and x in stat_slots (1..64) slots, added in slot order.
   * colsum[j] = alpha sum_k B[j, k] and colbias[j] = sum_k b_k W[j, k] (b the LayerNorm shift),
   * fp32 with at least 512 entries of padding past the last B row.  Not with SGD_EPI_DELTA. */
  int norm;
  const float* rstat;
  int stat_slots, stat_ld;
  float norm_eps;
  const float* colsum;
  const float* colbias;
  /* Writer of the residual stream (SGD_EPI_DELTA, or SGD_EPI_F32 writing h): with h16 set,
   * also stores fp16(new h) in h16 (row stride ldh, or ldo for F32) and, per row, the partial
   * sums of its new values' squares and values over the columns of each half of each output
   * tile in slot 2 t + half of stat_out (same layout as rstat, stat_out_ld >= M): the
   * statistics a following SGD_FNORM_* GEMM reads.  The slot count is 2 ceil(N / tile
   * width); sgd_kernel_gemm_stat_slots returns it. */
  void* h16;
  float* stat_out;
  int stat_out_ld;
  /* Optional, with h16: the CTA that completes the last column tile of a 128-row block
   * (tickets in stat_cnt, one int per row block, zero before the launch and left zero after
   * it; no CTA waits for another) adds that block's slots in slot order and stores each row's
   * totals in slot 0 of stat_final (same layout as rstat, 256-byte aligned like any device
   * allocation), so that a following SGD_FNORM_* GEMM reads stat_slots = 1 of stat_final. */
  int* stat_cnt;
  float* stat_final;
} sgd_epilogue_args;

/* Partial-sum slots a residual writer with these arguments fills (see h16 above). */
SGD_API int sgd_kernel_gemm_stat_slots(int M, int N, int K, const sgd_epilogue_args* epi,
                                       int variant, int* slots);

/*
 * C = alpha A B^T.  A fp16 [M, K] (row stride lda elements), B fp16 [N or 2N, K]
 * (row stride ldb).  K, lda, ldb multiples of 8; N multiple of 8; pointers 16-byte
 * aligned.  use_simt = 1 runs the plain SIMT kernel (reference / debugging), 0 the
 * tcgen05 + TMA kernel (M = 128, N = 256, K = 16 instructions, fp32 accumulators in
 * TMEM) with 64-element K-blocks, choosing by itself 128 x 256 or 128 x 128 tiles, 4 or 8
 * epilogue warps, and whether the tiles left over after the last full wave of CTAs are
 * split along K over all SMs ("stream-K": fp32 partial tiles in a workspace, summed in a
 * fixed order by the CTA that finishes a tile last, so results are deterministic); 3 the
 * form of 0 with 32-element K-blocks (64-byte swizzle); 2 and 4 are not defined and are
 * rejected with SGD_ERR_ARG; 5, 6, 7 force 128 x 256 tiles with 4 epilogue warps, 128 x 256 with 8, and
 * 128 x 128 with 8 and no stream-K (128 x 128 applies to plain, GELU and DELTA epilogues
 * only); 8 is 0 without stream-K, 9 is 0 with stream-K whenever the last wave is partial;
 * 10 forces 128 x 224 tiles (5 pipeline stages, no stream-K; plain, GELU and DELTA only);
 * 11 and 12 are 0 with the tiles visited M-fastest, and in groups of 16 row-blocks (each
 * group column by column, every other group backwards), instead of the choice made by 0
 * (groups where there are at least two groups and two waves).
 * The stream-K workspace is owned by the library, one per (device, stream), allocated
 * or grown by the first call that needs it (after synchronising that stream).
 */
SGD_API int sgd_kernel_gemm(const void* A, int lda, const void* B, int ldb, int M, int N, int K,
                    const sgd_epilogue_args* epi, int use_simt, void* stream);

/*
 * sgd_kernel_gemm without any device memory allocation.  The paper has no counterpart:
 * this is an interface for callers that cannot let the library allocate, such as a
 * process whose device memory is all reserved by its own pool allocator, or one that
 * cannot take the device-wide synchronisation that cudaMalloc / cudaFree may imply while
 * its other streams run.  Same arguments, variant codes (`variant` = use_simt above),
 * kernels and results bit for bit as sgd_kernel_gemm; the only difference is where a
 * stream-K split keeps its partial tiles and tile tickets: in one fixed array compiled
 * into the library (32 MiB of fp32 partial tiles, then 1024 tickets) instead of a
 * workspace the library allocates.
 * Limit: a problem whose stream-K split needs more than the array holds is rejected
 * with SGD_ERR_SHAPE before anything is launched (variant 8, or sgd_kernel_gemm, runs it).
 * The tickets are cleared (cudaMemsetAsync on `stream`) before each stream-K launch; the
 * partial tiles need no clearing (each is written before it is read within one launch).
 * Every call on a device uses the same array: calls that can overlap in time (launched
 * on different streams without ordering, or from several host threads at once) race on
 * it and can produce wrong results, so order them on one stream or with events.
 */
SGD_API int sgd_kernel_gemm_static_ws(const void* A, int lda, const void* B, int ldb, int M, int N,
                              int K, const sgd_epilogue_args* epi, int variant, void* stream);

/*
 * O = softmax(Q K^T / sqrt(d_head)) V per (sample, head), non-causal, keys beyond n_kv
 * masked.  Row r = b * n_q + i of q / o, row b * n_kv + j of k / v; head h occupies
 * columns [h d_head, (h+1) d_head).  fp16 in and out; d_head in {64, 72, 128};
 * leading dimensions in elements, multiples of 8.  impl = 0: tcgen05 for d_head 64 / 128
 * (S, P and O in TMEM; two 128-query tiles per CTA whose softmax warpgroups alternate with
 * each other's MMAs), the mma.sync kernel for 72 (see sgd_kernel_attention_hs for 72 on
 * tcgen05); 1: the mma.sync kernel for every d_head;
 * 2: tcgen05 with one query tile per CTA and P in shared memory; 3: the same as 0.
 */
SGD_API int sgd_kernel_attention(const void* q, int ldq, const void* k, const void* v, int ldkv,
                         void* o, int ldo, int batch, int n_q, int n_kv, int n_heads,
                         int d_head, int impl, void* stream);

/*
 * sgd_kernel_attention with the input heads `head_stride` columns apart (head h of q, k, v
 * at columns [h head_stride, h head_stride + d_head); head_stride >= d_head, a multiple of
 * 8); o keeps d_head columns per head.  With d_head 72, impl 0 / 3 run the tcgen05 kernel
 * when head_stride >= 80: each head is read as 80 columns (one 64-column and one
 * 16-column block), so columns [72, 80) after every Q head must be zero and those after
 * every K and V head finite (a layout whose gaps are zero, as sgd_step uses, satisfies
 * both); with head_stride 72 they fall back to the mma.sync kernel.
 */
SGD_API int sgd_kernel_attention_hs(const void* q, int ldq, const void* k, const void* v, int ldkv,
                                    int head_stride, void* o, int ldo, int batch, int n_q, int n_kv,
                                    int n_heads, int d_head, int impl, void* stream);

/*
 * out fp16 [rows, d] = norm(h fp32 [rows, d]); kind = sgd_norm_kind.  g, b: bf16 [d]
 * (NULL allowed for LN_PLAIN).  shift/scale: optional fp32 AdaLN modulation
 * [B, ld_mod]: out = norm(h) * (1 + scale[r / rows_per_batch]) + shift[...].
 * h 16-byte and out 8-byte aligned (else SGD_ERR_ARG).
 */
SGD_API int sgd_kernel_norm(const float* h, void* out, int rows, int d, int kind, const void* g,
                    const void* b, const float* shift, const float* scale, int ld_mod,
                    int rows_per_batch, float eps, void* stream);

/*
 * h fp32 [n] += sum_{i < n_caches} caches[i] (fp16 [n]), summed in order i = 0, 1, ...
 * in fp32.  caches_host: host array of n_caches (<= 96) device pointers.  n multiple
 * of 8, pointers 16-byte aligned.
 */
SGD_API int sgd_kernel_frozen_run(float* h, const void* const* caches_host, int n_caches, int64_t n,
                          void* stream);

/* Device status word shared by all kernels (bounded-wait expiry); returns and clears it. */
SGD_API int sgd_kernel_status(int* status_host);

/* *clamped_host = 1 if any kernel stored an fp16 value that it had to clamp to +-65504
 * (the value was out of fp16's range, or NaN) since the last call, else 0; clears the
 * flags.  A reading aid for fp16 operands, which the paper (bf16) does not use. */
SGD_API int sgd_kernel_f16_clamped(int* clamped_host);

/*
 * Failure-path self-test (no counterpart in the paper): launches on `stream` one kernel
 * whose thread waits, with the same bounded wait every kernel uses, on an mbarrier that
 * nothing completes.  After the wait limit (2 s) it records SGD_SELFTEST_TIMEOUT_CODE in
 * the device status word (read and cleared by sgd_kernel_status) and returns, leaving the
 * context usable.  Nothing faults, traps or hangs.
 */
#define SGD_SELFTEST_TIMEOUT_CODE 99
SGD_API int sgd_selftest_wait_timeout(void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SGD_KERNELS_H */
