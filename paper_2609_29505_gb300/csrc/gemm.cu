// Host side of the tcgen05 GEMM (planning: tile shape, tile order, stream-K split, tensor
// maps; dispatch to the kernel instantiations), the SIMT reference GEMM, the device status
// word and the fixed scratch of the allocation-free entry.  The kernel itself is in
// gemm_kernel.cuh.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "gemm_kernel.cuh"

namespace sgd {

using namespace gk;

__device__ int g_status;  // device status word (bounded-wait expiry codes)

// The tcgen05 kernels are instantiated in the gemm_tc_*.cu units.
namespace gk {
#define SGD_GEMM_EXTERN(FEAT)                                                                    \
  extern template cudaError_t launch_tc<64, 256, 8, FEAT>(const GemmPlan&, const TcArgs&, cudaStream_t); \
  extern template cudaError_t launch_tc<64, 256, 4, FEAT>(const GemmPlan&, const TcArgs&, cudaStream_t); \
  extern template cudaError_t launch_tc<64, 224, 8, FEAT>(const GemmPlan&, const TcArgs&, cudaStream_t); \
  extern template cudaError_t launch_tc<64, 128, 8, FEAT>(const GemmPlan&, const TcArgs&, cudaStream_t); \
  extern template cudaError_t launch_tc<32, 256, 8, FEAT>(const GemmPlan&, const TcArgs&, cudaStream_t);
SGD_GEMM_EXTERN(kFeatPlain)
SGD_GEMM_EXTERN(kFeatRms)
SGD_GEMM_EXTERN(kFeatLn)
SGD_GEMM_EXTERN(kFeatH16)
#undef SGD_GEMM_EXTERN
}  // namespace gk

namespace {

// ----------------------------------------------------------------------------
// SIMT reference GEMM: one output element per thread, fp32 accumulation in K order.
// ----------------------------------------------------------------------------

struct SimtArgs {
  const f16* A;
  int lda;
  const f16* B;
  int ldb;
  int M, N, K;
  EpiParams epi;
};

__device__ __forceinline__ float dot_f16(const f16* a, const f16* b, int K) {
  float acc = 0.f;
  int k = 0;
  for (; k + 8 <= K; k += 8) {
    float fa[8], fb[8];
    unpack_f16x8(*reinterpret_cast<const uint4*>(a + k), fa);
    unpack_f16x8(*reinterpret_cast<const uint4*>(b + k), fb);
#pragma unroll
    for (int i = 0; i < 8; ++i) acc = fmaf(fa[i], fb[i], acc);
  }
  for (; k < K; ++k) acc = fmaf(__half2float(a[k]), __half2float(b[k]), acc);
  return acc;
}

__global__ void gemm_simt_kernel(const SimtArgs a) {
  pdl_wait_and_trigger();
  const int col = blockIdx.x * blockDim.x + threadIdx.x;
  const int row = blockIdx.y;
  if (col >= a.N || row >= a.M) return;
  const EpiParams& e = a.epi;
  void* out = e.out_slot ? *e.out_slot : e.out;
  const f16* arow = a.A + static_cast<int64_t>(row) * a.lda;
  float v = dot_f16(arow, a.B + static_cast<int64_t>(col) * a.ldb, a.K) * e.alpha;
  switch (e.kind) {
    case SGD_EPI_GATED: {
      const float u = dot_f16(arow, a.B + static_cast<int64_t>(a.N + col) * a.ldb, a.K) * e.alpha;
      v = e.act ? v * gelu_erf_f(u) : silu_f(v) * u;
      break;
    }
    case SGD_EPI_GELU:
      v = e.act ? gelu_erf_f(v) : gelu_tanh_f(v);
      break;
    case SGD_EPI_ROPE:
      if (col < e.rope_cols) {
        const int half = e.d_head >> 1;
        const int i = col % e.d_head;
        const int pos = row % e.rope_tokens;
        const int partner = i < half ? col + half : col - half;
        const int fi = i < half ? i : i - half;
        const float c_ = e.rope_cos[pos * half + fi], s_ = e.rope_sin[pos * half + fi];
        const float p = dot_f16(arow, a.B + static_cast<int64_t>(partner) * a.ldb, a.K) * e.alpha;
        v = i < half ? v * c_ - p * s_ : v * c_ + p * s_;
      }
      break;
    case SGD_EPI_DELTA: {
      if (e.gate) v *= e.gate[static_cast<int64_t>(row / e.rows_per_batch) * e.ld_gate + col];
      float* hp = e.h + static_cast<int64_t>(row) * e.ldh + col;
      *hp = *hp + v;
      if (e.cache) e.cache[static_cast<int64_t>(row) * e.ld_cache + col] = __float2half_rn(sat_f16(v));
      return;
    }
    default:
      break;
  }
  const int oc = (e.kind == SGD_EPI_F16 && e.pad_src) ? (col / e.pad_src) * e.pad_dst + col % e.pad_src : col;
  if (e.kind == SGD_EPI_F32)
    reinterpret_cast<float*>(out)[static_cast<int64_t>(row) * e.ldo + col] = v;
  else
    reinterpret_cast<f16*>(out)[static_cast<int64_t>(row) * e.ldo + oc] = __float2half_rn(sat_f16(v));
}

// ----------------------------------------------------------------------------
// host side
// ----------------------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

}  // namespace

// fp16 [rows, cols] with row stride ld elements; box = box_cols (64, 32 or 16) columns x
// box_rows rows, 128- or 64-byte swizzle to match, out-of-range elements read as zero.
bool make_tmap_f16(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows,
                   int box_cols) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_cols), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  box_cols == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                 : (box_cols == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B),
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

int num_sms() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// ----------------------------------------------------------------------------
// Static stream-K scratch of sgd_kernel_gemm_static_ws: callers of that entry cannot
// have the library allocate device memory, so its stream-K partial tiles and tickets
// live in this fixed array instead: kStaticWsBytes of fp32 partials (enough for the
// 4096 x 4096 projections at K >= 3072 on 152 SMs, 56 tiles x 4 segments x 128 KB), then
// kStaticTickets tile tickets.  The array is zero when the module loads; the entry
// clears the tickets before each launch and the partials need no clearing.
// ----------------------------------------------------------------------------
constexpr size_t kStaticWsBytes = static_cast<size_t>(32) << 20;
constexpr int kStaticTickets = 1024;
static __device__ __align__(256) uint8_t g_static_scratch[kStaticWsBytes + kStaticTickets * sizeof(int)];

int gemm_static_scratch(float** ws, size_t* ws_floats, int** tickets, int* n_tickets, const char** why) {
  constexpr int kMaxDevices = 64;
  static std::mutex mu;
  static uint8_t* addr[kMaxDevices] = {nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *why = "gemm: no current CUDA device";
    return -1;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (!addr[dev]) {
    // once per device, with that device current (the symbol has one instance per device)
    void* q = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&q, g_static_scratch);
    if (e != cudaSuccess || !q) {
      *why = "gemm: cudaGetSymbolAddress of the static stream-K scratch failed";
      return -1;
    }
    addr[dev] = static_cast<uint8_t*>(q);
  }
  *ws = reinterpret_cast<float*>(addr[dev]);
  *ws_floats = kStaticWsBytes / sizeof(float);
  *tickets = reinterpret_cast<int*>(addr[dev] + kStaticWsBytes);
  *n_tickets = kStaticTickets;
  return 0;
}

int* device_status_ptr() {
  static int* ptr[64] = {nullptr};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return nullptr;
  if (!ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
    ptr[dev] = static_cast<int*>(p);
  }
  return ptr[dev];
}

// Stream-K split of the tiles left after the last full wave of `sms` CTAs: their
// tiles * num_k K iterations go to up to `sms` CTAs, at least a third of a tile's K range
// each, so that no tile is shared by more than kMaxSeg = 4 CTAs.  Measured on GB300 under
// its power cap, the split pays only where the last wave leaves much of the GPU idle
// (>= 12% of the tile slots of the launch), K is long enough (>= 48 K-blocks) for the
// partial stores and sums to be small next to a tile, and at least one full wave of
// data-parallel tiles follows to hide them; `force` takes any valid split.  max_seg:
// most CTAs sharing a tile, with the kernel's owner arithmetic.
struct SkSplit {
  int tiles = 0, ctas = 0, max_seg = 0;
};

SkSplit sk_split(int num_tiles, int num_k, int sms, bool force = false) {
  SkSplit r;
  const int rem = num_tiles % sms;
  if (rem == 0 || num_k < 2) return r;
  const int total = rem * num_k;
  const int min_iters = (num_k + 2) / 3;
  const int ctas = std::min(sms, total / min_iters);
  if (ctas <= rem) return r;
  const int slots = (num_tiles / sms + 1) * sms;
  const bool gain = num_k >= 48 && num_tiles >= sms && (slots - num_tiles) >= 0.12 * slots;
  if (!gain && !force) return r;
  auto owner = [&](int64_t i) { return static_cast<int>(((i + 1) * ctas - 1) / total); };
  int max_seg = 0;
  for (int t = 0; t < rem; ++t) {
    const int nseg = owner(static_cast<int64_t>(t) * num_k + num_k - 1) - owner(static_cast<int64_t>(t) * num_k) + 1;
    max_seg = std::max(max_seg, nseg);
  }
  if (max_seg > kMaxSeg) return r;
  r.tiles = rem;
  r.ctas = ctas;
  r.max_seg = max_seg;
  return r;
}

int gemm_plan(GemmPlan& p, const char** why) {
  const EpiParams& e = p.epi;
  const bool gated = e.kind == SGD_EPI_GATED;
  if (!p.A || !p.B || p.M <= 0 || p.N <= 0 || p.K <= 0) {
    *why = "gemm: null operand or empty shape";
    return -1;
  }
  if ((p.K % 8) || (p.lda % 8) || (p.ldb % 8) || (p.N % 8) || !aligned16(p.A) || !aligned16(p.B)) {
    *why = "gemm: K, lda, ldb, N must be multiples of 8 and operands 16-byte aligned";
    return -2;
  }
  if (e.kind == SGD_EPI_DELTA) {
    if (!e.h || (e.ldh % 4) || !aligned16(e.h) || (e.cache && (e.ld_cache % 8)) ||
        (e.gate && (e.ld_gate % 4 || e.rows_per_batch <= 0))) {
      *why = "gemm: DELTA epilogue needs an aligned residual (ldh % 4), ld_cache % 8, ld_gate % 4";
      return -2;
    }
  } else if (!e.out && !e.out_slot) {
    *why = "gemm: missing output";
    return -1;
  } else if (e.ldo % 8) {
    *why = "gemm: ldo must be a multiple of 8";
    return -2;
  }
  if (e.kind == SGD_EPI_ROPE &&
      (!(e.d_head == 64 || e.d_head == 128) || !e.rope_cos || !e.rope_sin || e.rope_tokens <= 0 ||
       (e.rope_cols % e.d_head))) {
    *why = "gemm: RoPE epilogue needs d_head 64 or 128 and cos/sin tables";
    return -2;
  }
  if (e.norm != SGD_FNORM_NONE) {
    if (e.norm != SGD_FNORM_RMS && e.norm != SGD_FNORM_LN) {
      *why = "gemm: bad folded-norm kind";
      return -1;
    }
    if (!e.rstat || e.stat_slots < 1 || e.stat_slots > kStatSlots || e.stat_ld < p.M ||
        (e.norm == SGD_FNORM_LN && (!e.colsum || !e.colbias)) || e.kind == SGD_EPI_DELTA) {
      *why = "gemm: folded norm needs row statistics (1..64 slots, stat_ld >= M), LN column "
             "vectors, and a non-residual epilogue";
      return -2;
    }
  }
  if (e.stat_cnt && (!e.h16 || !e.stat_final || !aligned16(e.stat_final))) {
    *why = "gemm: row-statistics finalisation needs the residual writer and a final buffer";
    return -2;
  }
  if (e.norm == SGD_FNORM_LN && e.kind == SGD_EPI_ROPE) {
    *why = "gemm: a folded LayerNorm has no RoPE epilogue (RoPE models use RMSNorm)";
    return -2;
  }
  if (e.norm != SGD_FNORM_NONE && e.h16) {
    *why = "gemm: a folded-norm GEMM cannot also write the residual stream";
    return -2;
  }
  if (e.pad_src) {
    if (e.kind != SGD_EPI_F16 || e.pad_src % 8 || e.pad_dst < e.pad_src || e.pad_dst % 8 ||
        e.ldo < ((p.N + e.pad_src - 1) / e.pad_src) * e.pad_dst) {
      *why = "gemm: head padding needs an F16 epilogue, pad_src and pad_dst multiples of 8, and ldo "
             "covering the padded width";
      return -2;
    }
  }
  if (e.h16) {
    if ((e.kind != SGD_EPI_DELTA && e.kind != SGD_EPI_F32) || e.gate || !e.stat_out || e.stat_out_ld < p.M ||
        !aligned16(e.h16)) {
      *why = "gemm: the fp16 copy of h needs a DELTA (without gate) or F32 epilogue and a statistics buffer";
      return -2;
    }
  }
  if (p.simt) {
    if (e.norm != SGD_FNORM_NONE || e.h16) {
      *why = "gemm: the SIMT kernel has no folded norm";
      return -2;
    }
    return 0;
  }
  const int b_rows = gated ? 2 * p.N : p.N;
  if (p.bk != 64 && p.bk != 32) p.bk = 64;
  const int num_m = (p.M + kBM - 1) / kBM;
  const int sms = num_sms();
  const int num_k = (p.K + p.bk - 1) / p.bk;
  // tile shape: 128-column tiles when they need clearly fewer tile-times than 256-column
  // tiles (a 128-column tile takes half the time of a 256-column one, at about 3/4 of its
  // efficiency, so: 2 * waves_128 < 3 * waves_256) and stream-K does not already even out
  // the last wave; they need a plain epilogue and one-CTA launches.
  const bool small_ok = !gated && e.kind != SGD_EPI_ROPE && p.bk == 64;
  // 128 x 224 tiles where they fill whole waves exactly, K is long and the last column of
  // tiles wastes under a tenth of N (e.g. M = N = 4096 at K >= 3072: 608 tiles = 4 waves;
  // measured 1266 against 1233 TFLOP/s for 128 x 256 with stream-K)
  const int n224 = (p.N + 223) / 224;
  if (p.bn == 0 && p.sk != 1 && small_ok && p.K >= 3072 && (num_m * n224) % sms == 0 &&
      10 * (n224 * 224 - p.N) < p.N)
    p.bn = 224;
  if (p.bn == 0) {
    const int t256 = num_m * (gated ? (p.N + 127) / 128 : (p.N + 255) / 256);
    const int w256 = (t256 + sms - 1) / sms;
    const int w128 = (num_m * ((p.N + 127) / 128) + sms - 1) / sms;
    SkSplit sk256 = sk_split(t256, num_k, sms);
    const bool sk_on = p.sk != 0 && sk256.tiles > 0;
    p.bn = (small_ok && !sk_on && 2 * w128 < 3 * w256) ? 128 : 256;
  }
  if ((p.bn != 128 && p.bn != 224) || !small_ok) p.bn = 256;
  if (p.bn == 224) p.sk = 0;
  // 8 epilogue warps (two per TMEM lane quarter, staged stores) except for RoPE, whose
  // per-thread state needs the 4-warp kernel's registers, and long-K gated MLPs, whose
  // epilogue hides behind the main loop (device time per launch: gated 2048 x 5120 x 1280
  // 44.9 against 65.0 us with 4 warps, 4096 x 12288 x 4096 495 against 491 us; RoPE
  // 4096 x 12288 x 4096 259 against 305 us with 8)
  if (p.epiw == 0) p.epiw = (e.kind == SGD_EPI_ROPE || (gated && p.K >= 3072)) ? 4 : 8;
  if (p.bn == 128 || p.bn == 224 || p.bk == 32) p.epiw = 8;
  if (p.encode && (!make_tmap_f16(&p.tmap_a, p.A, p.M, p.K, p.lda, 128, p.bk) ||
                   !make_tmap_f16(&p.tmap_b, p.B, b_rows, p.K, p.ldb, p.bn == 224 ? 224 : 128, p.bk))) {
    *why = "gemm: cuTensorMapEncodeTiled failed (driver entry point unavailable or bad layout)";
    return -5;
  }
  const int num_n = gated ? (p.N + 127) / 128 : (p.N + p.bn - 1) / p.bn;
  if (e.h16 && 2 * num_n > kStatSlots) {
    *why = "gemm: too many column tiles for the row-statistics slots";
    return -2;
  }
  const int units = num_m * num_n;
  p.grid = units < sms ? units : sms;
  // tile order.  M-fastest keeps A (the activations) in L2 while B streams through once,
  // which is the least DRAM traffic whenever A fits in L2 with room to spare (QKV, up, head
  // and attention-output projections: A = 33.5 MB).  When neither operand fits (the down
  // projection: 100 MB each), groups of 16 row-blocks (a 152-tile wave spanning ~16 x 9.5
  // tiles, about balanced between A and B bytes) read less than M-fastest.
  if (p.group_m < 0) {
    const double a_bytes = 2.0 * p.M * p.K, b_bytes = 2.0 * b_rows * p.K;
    constexpr double kL2Resident = 48e6;  // of 129 MB of L2, split between two dies
    p.group_m = (num_m >= 32 && num_n >= 4 && units >= 2 * sms && a_bytes > kL2Resident &&
                 b_bytes > kL2Resident)
                    ? 16
                    : 0;
  }
  p.sk_tiles = p.sk_ctas = p.max_seg = 0;
  if (p.sk != 0) {
    const SkSplit k = sk_split(units, num_k, sms, p.sk == 1);
    if (k.tiles > 0) {
      p.sk_tiles = k.tiles;
      p.sk_ctas = k.ctas;
      p.max_seg = k.max_seg;
      p.grid = units >= sms ? sms : k.ctas;
    }
  }
  return 0;
}

size_t gemm_ws_floats(const GemmPlan& p) {
  return p.sk_tiles > 0 ? static_cast<size_t>(p.sk_tiles) * p.max_seg * kBM * p.bn : 0;
}

template <int FEAT>
cudaError_t launch_feat(const GemmPlan& p, const TcArgs& a, cudaStream_t s) {
  if (p.bk == 32) return launch_tc<32, 256, 8, FEAT>(p, a, s);
  if (p.bn == 128) return launch_tc<64, 128, 8, FEAT>(p, a, s);
  if (p.bn == 224) return launch_tc<64, 224, 8, FEAT>(p, a, s);
  return p.epiw == 4 ? launch_tc<64, 256, 4, FEAT>(p, a, s) : launch_tc<64, 256, 8, FEAT>(p, a, s);
}

cudaError_t gemm_launch(const GemmPlan& p, cudaStream_t s) {
  if (p.simt) {
    SimtArgs a{p.A, p.lda, p.B, p.ldb, p.M, p.N, p.K, p.epi};
    dim3 grid((p.N + 127) / 128, p.M);
    return launch_k(gemm_simt_kernel, grid, dim3(128), 0, s, a);
  }
  TcArgs a;
  memcpy(&a.tmap_a, &p.tmap_a, sizeof(CUtensorMap));
  memcpy(&a.tmap_b, &p.tmap_b, sizeof(CUtensorMap));
  a.epi = p.epi;
  a.epi.M = p.M;
  a.epi.N = p.N;
  a.M = p.M;
  a.N = p.N;
  a.K = p.K;
  a.gated = p.epi.kind == SGD_EPI_GATED;
  a.num_m = (p.M + kBM - 1) / kBM;
  a.num_n = a.gated ? (p.N + 127) / 128 : (p.N + p.bn - 1) / p.bn;
  a.num_k = (p.K + p.bk - 1) / p.bk;
  a.group_m = p.group_m;
  a.status = device_status_ptr();
  a.sk_tiles = p.sk_tiles;
  a.sk_ctas = p.sk_ctas;
  a.max_seg = p.max_seg;
  a.ws = p.ws_ref ? *p.ws_ref : nullptr;
  a.sk_cnt = p.cnt_ref ? *p.cnt_ref : nullptr;
  if (p.sk_tiles > 0 && (!a.ws || !a.sk_cnt)) return cudaErrorInvalidValue;
  const EpiParams& e = p.epi;
  const int feat = e.norm == SGD_FNORM_RMS ? kFeatRms
                   : (e.norm == SGD_FNORM_LN ? kFeatLn : (e.h16 ? kFeatH16 : kFeatPlain));
  switch (feat) {
    case kFeatRms: return launch_feat<kFeatRms>(p, a, s);
    case kFeatLn: return launch_feat<kFeatLn>(p, a, s);
    case kFeatH16: return launch_feat<kFeatH16>(p, a, s);
    default: return launch_feat<kFeatPlain>(p, a, s);
  }
}

}  // namespace sgd
