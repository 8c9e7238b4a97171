// Internal interface between the C ABI (api.cu) and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include <vector>

#include "../../include/sgd.h"
#include "../../include/sgd_kernels.h"

namespace sgd {

using bf16 = __nv_bfloat16;
using f16 = __half;

// Epilogue parameters as the kernels see them (mirror of sgd_epilogue_args plus the
// output-pointer slot used by captured graphs and the output extent).
struct EpiParams {
  int kind;
  float alpha;            // accumulator scale (undoes the power-of-two weight scale)
  void* out;
  int ldo;
  void* const* out_slot;  // device address holding the output pointer (overrides out)
  float* h;
  int ldh;
  f16* cache;
  int ld_cache;
  const float* gate;
  int ld_gate;
  int rows_per_batch;
  int act;
  const float* rope_cos;
  const float* rope_sin;
  int rope_tokens;
  int d_head;
  int rope_cols;
  int M;
  int N;  // output columns (gated: f)
  // Pre-norm folded into the GEMM (A = fp16 copy of the residual stream h, the norm gain
  // folded into B): per row, rstd (and for LayerNorm the mean) come from the partial row
  // sums the last writer of h left in `rstat`; accumulator column j (B row j) becomes
  // RMS: rstd * acc_j;  LN: rstd * (acc_j - mean * colsum_j) + colbias_j.
  int norm;               // SGD_FNORM_NONE / _RMS / _LN
  const float* rstat;     // partial sums: slot p of row r at rstat[p * stat_ld + r] (sum of
                          // squares), rstat[(kStatSlots + p) * stat_ld + r] (sum)
  int stat_slots;         // slots the writer of h filled
  int stat_ld;            // rows between slots (M)
  float norm_eps;
  float norm_inv_d;       // 1 / K
  const float* colsum;    // LN: alpha * sum_k B[j, k] per B row
  const float* colbias;   // LN: sum_k b_k W[j, k] per B row (the shift through the weight)
  // Writer of h (DELTA, and F32 with h16 set): also store fp16(h_new) in h16 (ld = ldh, or
  // ldo for F32) and the row's partial sums over this thread's columns in slot
  // 2 * n_blk + part of stat_out (part: which column half of the tile).
  f16* h16;
  float* stat_out;
  int stat_out_ld;
  // Optional finalisation by the writer: the CTA that completes the last column tile of a
  // 128-row block (ticket from stat_cnt[row block], zero between launches, put back to zero
  // by that CTA; no CTA waits) adds the block's slots in slot order and stores the row
  // totals in slot 0 of stat_final (same layout as rstat, ld stat_out_ld): a following
  // folded-norm GEMM then reads one slot instead of 2 ceil(N / tile width).
  int* stat_cnt;
  float* stat_final;
  // SGD_EPI_F16 only: output column c goes to (c / pad_src) pad_dst + c % pad_src (heads of
  // pad_src columns written pad_dst apart; the gaps are never written).  0 = off.
  int pad_src, pad_dst;
};

// Row-statistics buffer: kStatSlots slots of sums of squares, then kStatSlots of sums.
constexpr int kStatSlots = 64;
enum { SGD_FNORM_NONE = 0, SGD_FNORM_RMS = 1, SGD_FNORM_LN = 2 };

// A planned GEMM: operands, epilogue and prebuilt TMA descriptors.
struct GemmPlan {
  const f16* A = nullptr;
  int lda = 0;
  const f16* B = nullptr;
  int ldb = 0;
  int M = 0, N = 0, K = 0;   // N = output columns
  EpiParams epi{};
  bool simt = false;
  int bk = 64;               // K elements per stage: 64 (128-byte swizzle) or 32 (64-byte)
  int bn = 0;                // output columns per tile: 256, 128, or 0 = choose by tile count
  int epiw = 0;              // epilogue warps: 4, 8, or 0 = choose by epilogue kind
  int sk = -1;               // stream-K for the tiles after the last full wave: -1 choose, 0 off, 1 on
  bool encode = true;        // false: choose the tiling only (no tensor maps; operands unused)
  int group_m = -1;          // tile order: -1 choose, 0 M-fastest, G > 0 groups of G row-blocks
  CUtensorMap tmap_a;
  CUtensorMap tmap_b;
  int grid = 0;
  int sk_tiles = 0, sk_ctas = 0, max_seg = 0;  // stream-K split (set by gemm_plan)
  // stream-K workspace, read at launch time through these (so that a plan built before its
  // workspace exists stays valid): fp32 [gemm_ws_floats] and int [sk_tiles] tickets that
  // must be zero before the first launch; a launch leaves them zero when it completes.
  float* const* ws_ref = nullptr;
  int* const* cnt_ref = nullptr;
};

// Validates shapes and builds the tensor maps; returns an sgd_status.
int gemm_plan(GemmPlan& p, const char** why);
cudaError_t gemm_launch(const GemmPlan& p, cudaStream_t s);
// fp32 elements of stream-K workspace a planned GEMM needs (0: data-parallel only).
size_t gemm_ws_floats(const GemmPlan& p);
// The fixed stream-K scratch of the current device (partials, then tickets) and its
// capacity; returns 0, or -1 with `why` set when its address cannot be obtained.
int gemm_static_scratch(float** ws, size_t* ws_floats, int** tickets, int* n_tickets, const char** why);
int* device_status_ptr();  // device address of the shared status word
// Accessors of the fp16 clamp flags of every kernel translation unit (registered at load).
const std::vector<unsigned int* (*)()>& f16_clamp_flags();
int num_sms();
// 2-D fp16 tensor map: [rows, cols] with row stride ld elements, box 64 x box_rows,
// 128-byte swizzle (defined in gemm.cu).
bool make_tmap_f16(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows,
                   int box_cols = 64);

// Attention.
struct AttnParams {
  const f16* q;
  int ldq;
  const f16* k;
  const f16* v;
  int ldkv;
  f16* o;
  int ldo;
  int batch, n_q, n_kv, n_heads, d_head;
  int impl;  // 0: tcgen05 with two query tiles per CTA where d_head is 64 or 128 (72 from a
             //    head-padded layout), else mma.sync; 1: mma.sync; 2: tcgen05, one query
             //    tile per CTA; 3: same as 0
  int head_stride;  // input (q, k, v) columns between heads; 0 = d_head.  Outputs: d_head.
};
// A planned attention launch: parameters plus TMA descriptors for the tcgen05 kernel.
struct AttnPlan {
  AttnParams p{};
  bool tc = false;
  bool pp = false;  // two query tiles per CTA (attn_pp_kernel)
  CUtensorMap tmap_q;
  CUtensorMap tmap_kv;
  CUtensorMap tmap_v;
  CUtensorMap tmap_q16;  // d_h 72: 16-column boxes (32-byte swizzle)
  CUtensorMap tmap_k16;
  CUtensorMap tmap_v16;
};
int attn_check(const AttnParams& p, const char** why);
int attn_plan(AttnPlan& plan, const char** why);
cudaError_t attn_launch(const AttnPlan& plan, cudaStream_t s);

// Norm: out = norm(h) [* (1 + scale) + shift].
struct NormParams {
  const float* h;
  f16* out;
  int rows, d, kind;
  const bf16* g;
  const bf16* b;
  const float* shift;
  const float* scale;
  int ld_mod, rows_per_batch;
  float eps;
};
cudaError_t norm_launch(const NormParams& p, cudaStream_t s);

// Frozen run: h += sum caches (in cache order, fp32).  With h16 set, the rows are
// processed in chunks of kStatChunk columns (one warp per chunk) and each chunk also
// stores fp16(h) into h16 and its partial row sums into stat slot `chunk` (sum of squares,
// and the sum at kStatSlots + chunk); n_caches may then be 0 (statistics of h only).
constexpr int kMaxRun = 96;
constexpr int kStatChunk = 1024;
struct FrozenParams {
  float* h;
  const f16* caches[kMaxRun];
  int n_caches;
  int64_t n;
  int rows, d;       // row structure (used with h16)
  f16* h16;
  float* stat;       // [2 kStatSlots][rows]
};
cudaError_t frozen_launch(const FrozenParams& p, cudaStream_t s);
inline int frozen_stat_slots(int d) { return (d + kStatChunk - 1) / kStatChunk; }

// Lagged-drift reduction of the input-aware policy (App. B.1) for one scheduled group:
// partial[b] = (sum (h - snap)^2, sum h^2) over block b's elements (fp32, fixed order),
// then snap = h.  n % 4 == 0, 16-byte aligned.  drift_reduce sums each group's kDriftBlocks
// partials in a fixed order, in double: sums[2 g], sums[2 g + 1].
constexpr int kDriftBlocks = 1024;
struct DriftParams {
  const float* h;
  float* snap;
  int64_t n;
  float* partial;  // [kDriftBlocks][2]
};
cudaError_t drift_launch(const DriftParams& p, cudaStream_t s);
// One thread waits (bounded) on an mbarrier nothing completes and records `code`.
cudaError_t wait_selftest_launch(int* status, int code, cudaStream_t s);
cudaError_t drift_reduce_launch(const float* partials, int n_groups, double* sums, cudaStream_t s);

// Per-step I/O slot (device memory) read by graph kernels.
struct IoSlot {
  const void* state;
  void* out;
  const int32_t* class_ids;
  const void* ctx;
  float t;
  int step;
};
cudaError_t io_set_launch(IoSlot* slot, const IoSlot& v, cudaStream_t s);

// Small always-on pieces (stem, conditioning, heads).
struct StemParams {
  int kind;
  const IoSlot* slot;
  float* h;
  int batch, n_tokens, n_prefix, d, d_in;
  const bf16* w_stem;
  const bf16* pos;
  const bf16* class_emb;
  const bf16* embed;
  int vocab, n_classes;  // ids are clamped into [0, vocab) / [0, n_classes)
};
cudaError_t stem_launch(const StemParams& p, cudaStream_t s);

// out[r, j] = sum_k act(x[r, k]) W[j, k] (+ add[r, j]); x fp32 or computed on the fly.
constexpr int kGemvMaxSeg = 64;
struct GemvParams {
  float* out;
  int ldo;
  const float* x;      // [rows, K] fp32 (ignored when x_sinusoid)
  int ldx;
  int x_sinusoid;      // x = sinusoid(t, K) from the slot, one row
  const IoSlot* slot;
  int in_silu;         // act = silu
  const bf16* W;       // [N, K]
  int N, K, rows;
  const bf16* add_class;  // optional: + class_emb[class_ids[r]] (bf16 [n_classes, N])
  int n_classes;          // class ids are clamped into [0, n_classes)
  const float* add_vec;   // optional: + add_vec[j] (broadcast over rows)
  float* out_silu;        // optional: silu(out) written alongside (same layout)
  // n_seg > 0: n_seg independent products with the same x, N, K and ldo in one launch
  // (W = w_seg[i], out = out_seg[i]; W and out above are ignored) -- the AdaLN modulation
  // of every block a step runs
  int n_seg;
  const bf16* w_seg[kGemvMaxSeg];
  float* out_seg[kGemvMaxSeg];
};
cudaError_t gemv_launch(const GemvParams& p, cudaStream_t s);

// Row-wise small-N linear for heads: out[r, j] = norm(h[r]) . W[j] for j < N (N <= 64); the
// norm (RMSNorm, LayerNorm, or LayerNorm without affine then the AdaLN modulation
// x (1 + scale_b) + shift_b) is computed from the fp32 row in the same kernel.
struct HeadParams {
  const float* h;      // [rows_total, K] fp32 residual stream
  int ldx;
  int norm_kind;       // sgd_norm_kind
  const bf16* g;
  const bf16* b;
  const float* shift;  // AdaLN: [batch, ld_mod]
  const float* scale;
  int ld_mod;
  float eps;
  const bf16* W;       // [N, K]
  int N, K;
  int batch, n_tokens, n_prefix;  // rows r = b * n_tokens + n, n >= n_prefix are output
  int out_channels;               // columns written (<= N)
  const IoSlot* slot;             // out pointer: fp32 [batch, n_tokens - n_prefix, out_channels]
};
cudaError_t head_small_launch(const HeadParams& p, cudaStream_t s);

// Identity head: out (from slot) = h.
cudaError_t copy_out_launch(const IoSlot* slot, const float* h, int64_t n, cudaStream_t s);

// U-ViT: dst fp16 [rows, ld_dst] columns [col0, col0 + d) = fp16(h).
cudaError_t pack_f16_launch(f16* dst, int ld_dst, int col0, const float* h, int rows, int d,
                            cudaStream_t s);

// Weight preparation: max |w| of a bf16 tensor (into *out, device) and the exact
// conversion dst = fp16(w * 2^shift); also plain bf16 -> fp16 conversion (shift 0).
cudaError_t absmax_bf16_launch(const bf16* w, int64_t n, float* out, cudaStream_t s);
cudaError_t convert_bf16_f16_launch(const bf16* w, f16* dst, int64_t n, int shift, cudaStream_t s);
// Folded pre-norm gain: W[j, k] g[k] for a bf16 [rows, K] weight and bf16 gain [K] — the
// max |W g| (absmax, *out starting at 0) and the conversion dst = fp16(W g 2^shift).
cudaError_t absmax_scaled_launch(const bf16* w, const bf16* g, int64_t rows, int K, float* out,
                                 cudaStream_t s);
cudaError_t convert_scaled_launch(const bf16* w, const bf16* g, f16* dst, int64_t rows, int K, int shift,
                                  cudaStream_t s);
// out[j] = scale * sum_k W[j, k] x[k] per row j of an fp16 (x = 1) or bf16 (x bf16 [K])
// [rows, K] matrix, accumulated in double.
cudaError_t rowsum_f16_launch(const f16* w, int64_t rows, int K, float scale, float* out, cudaStream_t s);
cudaError_t rowdot_bf16_launch(const bf16* w, const bf16* x, int64_t rows, int K, float* out,
                               cudaStream_t s);

cudaError_t sampler_launch(float* z, const float* eps, float alpha, float beta, int64_t n,
                           cudaStream_t s);

}  // namespace sgd
