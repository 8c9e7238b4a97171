// The tcgen05 GEMM kernel (C = A B^T with fused epilogues), shared by the translation units
// that instantiate it: gemm_tc_plain.cu, gemm_tc_rms.cu, gemm_tc_ln.cu and gemm_tc_h16.cu,
// one per epilogue feature set (FEAT), compiled in parallel; gemm.cu plans and dispatches.
//
// This is the projection kernel of every active residual branch (Algorithm 2: an
// active unit computes Delta = F_l(h; c), refreshes its cache and adds Delta to the
// residual stream).  The branch's last projection runs with the DELTA epilogue,
// which stores the fp16 cache entry and adds Delta to the fp32 residual h in the
// same pass over the tile.  Operands are fp16 (weights converted exactly from bf16
// with a power-of-two scale, undone by `alpha`), accumulation is fp32 in TMEM.
//
// Design (one CTA per SM, persistent over 128 x 256 output tiles):
//   warp 0      TMA producer: A box 128x64 and two B boxes 128x64 per stage into a
//               4-stage ring of 48 KB stages (128-byte swizzle).
//   warp 1      allocates 512 TMEM columns (two 128x256 fp32 accumulators) and one
//               elected lane issues tcgen05.mma (M=128, N=256, K=16) four times per
//               stage, committing each stage back to the producer.
//   warps 2-9   epilogue: tcgen05.ld rows out of TMEM (warp w owns TMEM lanes
//               32 (w % 4) ..., warps w and w + 4 split the tile's columns), apply the
//               epilogue, store to global memory.  The two accumulators let the epilogue
//               of tile i overlap the MMAs of tile i+1.
// Every wait is bounded (common.cuh); on expiry the CTA drains its own copies and
// MMAs, frees TMEM and exits with the device status word set.
//
// FEAT (compile-time epilogue features, so that each kernel carries only its own code and
// registers): kFeatPlain; kFeatRms / kFeatLn, the pre-norm folded into the GEMM
// (EpiParams::norm); kFeatH16, a writer of the residual stream that also emits fp16(h) and
// the row sums (EpiParams::h16).
#pragma once

#include <cstring>

#include "common.cuh"
#include "kernels.h"

namespace sgd {
namespace gk {


constexpr int kBM = 128;

enum { kFeatPlain = 0, kFeatRms = 1, kFeatLn = 2, kFeatH16 = 3 };

// K-block geometry.  BK = 64: 128-byte rows, 128-byte swizzle, 4 stages of 48 KB.
// BK = 32: 64-byte rows, 64-byte swizzle, 9 stages of 24 KB — the same MMA work per
// byte but a third more bytes in flight, to cover more of the TMA refill latency.
// BN = 256, 224 or 128 accumulator columns per tile (two accumulators in TMEM); EPIW = 4 or
// 8 epilogue warps (8: warps w and w + 4 split the tile's columns).  BN = 224 tiles N = 4096
// into 19 columns of tiles (608 tiles = 4 full waves of 152 at M = 4096) and its 44 KB stages
// fit 5 deep.
template <int BK, int BN = 256, int EPIW = 8>
struct TileCfg {
  static constexpr int kBK = BK;
  static constexpr int kBN = BN;
  static constexpr int kEpiWarps = EPIW;
  static constexpr int kThreads = 64 + 32 * EPIW;
  static constexpr int kTmemCols = BN == 224 ? 512 : 2 * BN;  // allocations are powers of 2
  static constexpr int kTileA = kBM * BK * 2;
  static constexpr int kTileBHalf = 128 * BK * 2;
  static constexpr int kTileB = BN * BK * 2;
  static constexpr int kStageBytes = kTileA + kTileB;
  // epilogue staging: 4 KB per epilogue warp (32 rows x 32 fp32 columns) for the residual
  // epilogue's coalesced read-modify-write of h; none at BN 224, whose 5 stages fill the rest,
// nor in the 4-warp kernel
  static constexpr int kStaging = (BN == 224 || EPIW != 8) ? 0 : EPIW * 4096;
  static constexpr int kStages = BN == 224 ? 5 : (224 * 1024 - kStaging) / kStageBytes;
  static constexpr int kSmemBytes = kStages * kStageBytes + kStaging + 1024 /*align*/ + 256 /*barriers*/;
  static_assert(kSmemBytes <= 232448, "shared memory");
  static_assert((2 * kStages + 5) * 8 + 4 * 4 <= 256, "barrier block");
};

template <int BK>
__device__ __forceinline__ uint64_t operand_desc(uint32_t saddr) {
  return BK == 64 ? smem_desc_sw128(saddr) : smem_desc_sw64(saddr);
}

struct TcArgs {
  CUtensorMap tmap_a;
  CUtensorMap tmap_b;
  EpiParams epi;
  int M, N, K;  // N = output columns
  int num_m, num_n, num_k;
  int group_m;  // tile order: 0 = M-fastest; G = groups of G row-blocks, see tile_coords
  int gated;    // B second half starts at row N (= f)
  int* status;
  // stream-K (0 tiles: data-parallel only)
  int sk_tiles, sk_ctas, max_seg;
  float* ws;    // [sk_tiles][max_seg][128 * BN] fp32 partial accumulators (max_seg <= kMaxSeg)
  int* sk_cnt;  // [sk_tiles] tickets, zero between launches
};


// ----------------------------------------------------------------------------
// epilogue: 8 consecutive output columns of one row
// ----------------------------------------------------------------------------

__device__ __forceinline__ void store8_f16(void* base, int ld, int row, int col, const float* v) {
  f16* p = reinterpret_cast<f16*>(base) + static_cast<int64_t>(row) * ld + col;
  *reinterpret_cast<uint4*>(p) = pack_f16x8(v);
}

__device__ __forceinline__ void epi_store8(const EpiParams& e, void* out, int row, int col,
                                           float* v) {
  switch (e.kind) {
    case SGD_EPI_F16:
      store8_f16(out, e.ldo, row, e.pad_src ? (col / e.pad_src) * e.pad_dst + col % e.pad_src : col, v);
      break;
    case SGD_EPI_ROPE:
    case SGD_EPI_GATED:
      store8_f16(out, e.ldo, row, col, v);
      break;
    case SGD_EPI_GELU: {
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = e.act ? gelu_erf_f(v[i]) : gelu_tanh_f(v[i]);
      store8_f16(out, e.ldo, row, col, v);
      break;
    }
    case SGD_EPI_F32: {
      float4* p = reinterpret_cast<float4*>(reinterpret_cast<float*>(out) +
                                            static_cast<int64_t>(row) * e.ldo + col);
      p[0] = make_float4(v[0], v[1], v[2], v[3]);
      p[1] = make_float4(v[4], v[5], v[6], v[7]);
      break;
    }
    case SGD_EPI_DELTA: {
      if (e.gate) {
        const float4* g = reinterpret_cast<const float4*>(
            e.gate + static_cast<int64_t>(row / e.rows_per_batch) * e.ld_gate + col);
        const float4 g0 = g[0], g1 = g[1];
        v[0] *= g0.x; v[1] *= g0.y; v[2] *= g0.z; v[3] *= g0.w;
        v[4] *= g1.x; v[5] *= g1.y; v[6] *= g1.z; v[7] *= g1.w;
      }
      float4* hp = reinterpret_cast<float4*>(e.h + static_cast<int64_t>(row) * e.ldh + col);
      float4 h0 = hp[0], h1 = hp[1];
      h0.x += v[0]; h0.y += v[1]; h0.z += v[2]; h0.w += v[3];
      h1.x += v[4]; h1.y += v[5]; h1.z += v[6]; h1.w += v[7];
      hp[0] = h0;
      hp[1] = h1;
      if (e.cache) store8_f16(e.cache, e.ld_cache, row, col, v);
      break;
    }
    default:
      break;
  }
}

__device__ __forceinline__ void u32_to_f32x16(const uint32_t* r, float* f, float alpha) {
#pragma unroll
  for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(r[i]) * alpha;
}

// Accumulator sources for the epilogue.  load2(c0, c1, x, y) returns alpha times the
// accumulator at tile columns [c0, c0 + 16) and [c1, c1 + 16) of this thread's row.
// TmemSrc reads the tile's TMEM accumulator; every lane of the warp must call it together
// (tcgen05.ld is .sync.aligned).
struct TmemSrc {
  uint32_t tbase;
  float alpha;
  __device__ __forceinline__ void load2(int c0, int c1, float* x, float* y) const {
    uint32_t r0[16], r1[16];
    tmem_ld16(tbase + c0, r0);
    tmem_ld16(tbase + c1, r1);
    tmem_ld_wait16(r0);
    tmem_ld_wait16(r1);
    u32_to_f32x16(r0, x, alpha);
    u32_to_f32x16(r1, y, alpha);
  }
};

// Stream-K partial tiles in the workspace: slot j of a tile holds the raw fp32
// accumulator of its j-th K segment (at most kMaxSeg segments), laid out
// [BN / 4][128 rows] x float4 so that a warp's 32 rows are one contiguous 512-byte run.
// WsSrc, used by the CTA that finishes a tile, adds the slots in slot order (a fixed
// order, so the result does not depend on which CTA finishes last), loading two slots
// at a time.
constexpr int kMaxSeg = 4;

template <int BN>
struct WsSrc {
  const float* slot0;
  int nseg;
  int r;  // row within the tile
  float alpha;
  __device__ __forceinline__ void load16(int c, float* x) const {
    const float4* p = reinterpret_cast<const float4*>(slot0) + (c >> 2) * kBM + r;
    constexpr size_t kSlot = static_cast<size_t>(kBM) * BN / 4;  // float4 per slot
#pragma unroll
    for (int i = 0; i < 16; ++i) x[i] = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxSeg; j += 2) {
      if (j < nseg) {
        // the second slot's loads are unconditional (a predicated load makes the compiler
        // spill); past the last slot they repeat the first slot's addresses, unused
        const int j1 = j + 1 < nseg ? j + 1 : j;
        float4 u[4], w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          u[i] = __ldcg(p + j * kSlot + i * kBM);
          w[i] = __ldcg(p + j1 * kSlot + i * kBM);
        }
        const bool two = j + 1 < nseg;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          x[4 * i] += u[i].x;
          x[4 * i + 1] += u[i].y;
          x[4 * i + 2] += u[i].z;
          x[4 * i + 3] += u[i].w;
          x[4 * i] = two ? x[4 * i] + w[i].x : x[4 * i];
          x[4 * i + 1] = two ? x[4 * i + 1] + w[i].y : x[4 * i + 1];
          x[4 * i + 2] = two ? x[4 * i + 2] + w[i].z : x[4 * i + 2];
          x[4 * i + 3] = two ? x[4 * i + 3] + w[i].w : x[4 * i + 3];
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) x[i] *= alpha;
  }
  __device__ __forceinline__ void load2(int c0, int c1, float* x, float* y) const {
    load16(c0, x);
    load16(c1, y);
  }
};

// Store the raw TMEM accumulator columns [c0, c1) of this thread's row r into a
// workspace slot (layout of WsSrc).
template <int BN>
__device__ __forceinline__ void store_partial(float* slot, int r, uint32_t tbase, int c0, int c1) {
  uint32_t v0[16], v1[16];
  for (int c = c0; c < c1; c += 32) {
    tmem_ld16(tbase + c, v0);
    tmem_ld16(tbase + c + 16, v1);
    tmem_ld_wait16(v0);
    tmem_ld_wait16(v1);
    float4* p = reinterpret_cast<float4*>(slot) + (c >> 2) * kBM + r;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      __stcg(p + i * kBM, make_float4(__uint_as_float(v0[4 * i]), __uint_as_float(v0[4 * i + 1]),
                                      __uint_as_float(v0[4 * i + 2]), __uint_as_float(v0[4 * i + 3])));
#pragma unroll
    for (int i = 0; i < 4; ++i)
      __stcg(p + (4 + i) * kBM,
             make_float4(__uint_as_float(v1[4 * i]), __uint_as_float(v1[4 * i + 1]),
                         __uint_as_float(v1[4 * i + 2]), __uint_as_float(v1[4 * i + 3])));
  }
}

// Folded pre-norm (EpiParams::norm): the row's rstd and mean from the partial sums the
// last writer of h left, summed in slot order (the same order on every run).
struct RowNorm {
  float rstd, mean;
};

// Sum of `n` slots of a row's partial sums, slot order (the same bits on every run): eight
// loads are issued together and then added one after another (a zero past the last slot
// leaves the sum unchanged), instead of one load latency per slot.
__device__ __forceinline__ float sum_slots(const float* base, int64_t ld, int n) {
  float s = 0.f;
  for (int p = 0; p < n; p += 8) {
    float v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = (p + i < n) ? __ldcg(base + static_cast<int64_t>(p + i) * ld) : 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) s += v[i];
  }
  return s;
}

template <int FEAT>
__device__ __forceinline__ RowNorm row_norm(const EpiParams& e, int row, bool row_ok) {
  RowNorm n{1.f, 0.f};
  if constexpr (FEAT == kFeatRms || FEAT == kFeatLn) {
    const int r = row_ok ? row : 0;
    const float ss = sum_slots(e.rstat + r, e.stat_ld, e.stat_slots);
    if constexpr (FEAT == kFeatRms) {
      n.rstd = rsqrtf(ss * e.norm_inv_d + e.norm_eps);
    } else {
      const float s1 = sum_slots(e.rstat + static_cast<int64_t>(kStatSlots) * e.stat_ld + r, e.stat_ld,
                                 e.stat_slots);
      const double mean = static_cast<double>(s1) * e.norm_inv_d;
      const double var = fmax(static_cast<double>(ss) * e.norm_inv_d - mean * mean, 0.0);
      n.mean = static_cast<float>(mean);
      n.rstd = rsqrtf(static_cast<float>(var) + e.norm_eps);
    }
  }
  return n;
}

// Residual (DELTA) epilogue: pull this thread's part of the tile's h rows into L2 before
// waiting for the accumulator, so that the epilogue reads them from L2 (the wait is idle
// time; for a CTA's last tile no mainloop hides the DRAM latency otherwise).
__device__ __forceinline__ void prefetch_h_row(const EpiParams& e, int row, int M, int N, int n0, int cb,
                                               int ce) {
  if (e.kind != SGD_EPI_DELTA || row >= M) return;
  const int c1 = min(n0 + ce, N);
  const float* hr = e.h + static_cast<int64_t>(row) * e.ldh;
  for (int c = n0 + cb; c < c1; c += 32)  // 128-byte lines
    asm volatile("prefetch.global.L2 [%0];" ::"l"(hr + c));
}

// Apply the folded norm to 16 accumulator values whose B rows are brow .. brow + 15
// (colsum / colbias are padded past the last B row, so the loads need no guard).
template <int FEAT>
__device__ __forceinline__ void apply_norm16(const EpiParams& e, const RowNorm& n, int brow, float* v) {
  if constexpr (FEAT == kFeatRms) {
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] *= n.rstd;
  } else if constexpr (FEAT == kFeatLn) {
    const float4* cs = reinterpret_cast<const float4*>(e.colsum + brow);
    const float4* cb = reinterpret_cast<const float4*>(e.colbias + brow);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 u = cs[q], w = cb[q];
      v[4 * q] = n.rstd * (v[4 * q] - n.mean * u.x) + w.x;
      v[4 * q + 1] = n.rstd * (v[4 * q + 1] - n.mean * u.y) + w.y;
      v[4 * q + 2] = n.rstd * (v[4 * q + 2] - n.mean * u.z) + w.z;
      v[4 * q + 3] = n.rstd * (v[4 * q + 3] - n.mean * u.w) + w.w;
    }
  }
}

// Writer of h: the fp16 copy of 8 new values of h and their contribution to the row sums.
__device__ __forceinline__ void emit_h8(const EpiParams& e, int ld, int row, int col, const float* hv,
                                        float& ss, float& s1) {
  store8_f16(e.h16, ld, row, col, hv);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    ss = fmaf(hv[i], hv[i], ss);
    s1 += hv[i];
  }
}

__device__ __forceinline__ void emit_stats(const EpiParams& e, int row, int slot, float ss, float s1) {
  e.stat_out[static_cast<int64_t>(slot) * e.stat_out_ld + row] = ss;
  e.stat_out[static_cast<int64_t>(kStatSlots + slot) * e.stat_out_ld + row] = s1;
}

// Residual epilogue through this warp's 4 KB staging buffer `stg` (32 rows x 8 float4,
// 16-byte chunk j of row r at r * 8 + (j ^ (r & 7)), so that both access patterns below are
// free of bank conflicts).  Per 32-column chunk: the warp loads its 32 rows of h coalesced
// (8 lanes per 128-byte row segment), each thread adds its row's accumulator (times the
// AdaLN gate) in shared memory, and the warp stores h and the fp16 cache coalesced.  With
// one thread per row the same accesses touch 32 rows per instruction, which made the
// epilogue of a short-K projection take longer than its main loop.
template <class Src>
__device__ __forceinline__ void delta_staged(const TcArgs& a, int row, int n0, const Src& src, int cb, int ce,
                                             float4* stg) {
  const EpiParams& e = a.epi;
  const int lane = threadIdx.x & 31;
  const int row0 = row - lane;  // the warp's first row
  const int lr = lane >> 3, lc = lane & 7;
  const bool row_ok = row < a.M;
  const float* grow =
      e.gate ? e.gate + static_cast<int64_t>(row_ok ? row / e.rows_per_batch : 0) * e.ld_gate + n0 : nullptr;
#pragma unroll 1
  for (int c = cb; c < ce; c += 32) {
    const int col0 = n0 + c;
    if (col0 >= a.N) break;
    const bool c_ok = col0 + 4 * lc < a.N;  // this lane's float4 in the coalesced phases (N % 8 == 0)
    {
      float4 hv[8];
#pragma unroll
      for (int it = 0; it < 8; ++it) {
        const int r = row0 + it * 4 + lr;
        hv[it] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (r < a.M && c_ok)
          hv[it] = *reinterpret_cast<const float4*>(e.h + static_cast<int64_t>(r) * e.ldh + col0 + 4 * lc);
      }
#pragma unroll
      for (int it = 0; it < 8; ++it) {
        const int r = it * 4 + lr;
        stg[r * 8 + (lc ^ (r & 7))] = hv[it];
      }
    }
    __syncwarp();
    float x[16], y[16];
    src.load2(c, c + 16, x, y);
    if (grow) {  // columns past N (the tile's edge) read the row's last four, never stored
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        const float4 gv = *reinterpret_cast<const float4*>(grow + min(c + 4 * g, a.N - n0 - 4));
        float* v = g < 4 ? x + 4 * g : y + 4 * (g - 4);
        v[0] *= gv.x; v[1] *= gv.y; v[2] *= gv.z; v[3] *= gv.w;
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float* v = j < 4 ? x + 4 * j : y + 4 * (j - 4);
      float4& hs = stg[lane * 8 + (j ^ (lane & 7))];
      float4 h4 = hs;
      h4.x += v[0]; h4.y += v[1]; h4.z += v[2]; h4.w += v[3];
      hs = h4;
    }
    __syncwarp();
#pragma unroll
    for (int it = 0; it < 8; ++it) {
      const int r = it * 4 + lr;
      if (row0 + r < a.M && c_ok)
        *reinterpret_cast<float4*>(e.h + static_cast<int64_t>(row0 + r) * e.ldh + col0 + 4 * lc) =
            stg[r * 8 + (lc ^ (r & 7))];
    }
    if (e.cache) {
      __syncwarp();
      uint4* su = reinterpret_cast<uint4*>(stg);
#pragma unroll
      for (int j = 0; j < 4; ++j) su[lane * 8 + (j ^ (lane & 7))] = pack_f16x8(j < 2 ? x + 8 * j : y + 8 * (j - 2));
      __syncwarp();
      const int lr4 = lane >> 2, lc4 = lane & 3;
      const bool c8_ok = col0 + 8 * lc4 < a.N;
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int r = it * 8 + lr4;
        if (row0 + r < a.M && c8_ok)
          *reinterpret_cast<uint4*>(e.cache + static_cast<int64_t>(row0 + r) * e.ld_cache + col0 + 8 * lc4) =
              su[r * 8 + (lc4 ^ (r & 7))];
      }
    }
    __syncwarp();  // the next chunk overwrites the staging buffer
  }
}

// Coalesced stores through this warp's staging buffer (layout as in delta_staged): every
// thread puts 32 consecutive output values of its row (columns col0 .. col0 + 31), 16 at a
// time (put16 with half 0, then 1), and flush stores rows row0 .. row0 + 31.  fp16: 64
// bytes per row, stored as 4 lanes x 16 bytes per row (head-padded layouts remap each
// 8-column group); fp32: 128 bytes per row, 8 lanes per row.
__device__ __forceinline__ void stage_put16_f16(float4* stg, int half, const float* v) {
  const int lane = threadIdx.x & 31;
  uint4* su = reinterpret_cast<uint4*>(stg);
  su[lane * 8 + ((2 * half) ^ (lane & 7))] = pack_f16x8(v);
  su[lane * 8 + ((2 * half + 1) ^ (lane & 7))] = pack_f16x8(v + 8);
}

__device__ __forceinline__ void stage_flush_f16(const EpiParams& e, void* out, int row0, int M, int N, int col0,
                                                float4* stg) {
  const int lane = threadIdx.x & 31;
  const uint4* su = reinterpret_cast<const uint4*>(stg);
  __syncwarp();
  const int lr4 = lane >> 2, lc4 = lane & 3;
  const int col = col0 + 8 * lc4;
  const int dcol = e.pad_src ? (col / e.pad_src) * e.pad_dst + col % e.pad_src : col;
  f16* o = reinterpret_cast<f16*>(out);
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int r = it * 8 + lr4;
    if (row0 + r < M && col < N)
      *reinterpret_cast<uint4*>(o + static_cast<int64_t>(row0 + r) * e.ldo + dcol) = su[r * 8 + (lc4 ^ (r & 7))];
  }
  __syncwarp();  // the next chunk overwrites the staging buffer
}

__device__ __forceinline__ void stage_put16_f32(float4* stg, int half, const float* v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    stg[lane * 8 + ((4 * half + j) ^ (lane & 7))] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
}

__device__ __forceinline__ void stage_flush_f32(const EpiParams& e, void* out, int row0, int M, int N, int col0,
                                                float4* stg) {
  const int lane = threadIdx.x & 31;
  __syncwarp();
  const int lr = lane >> 3, lc = lane & 7;
  const int col = col0 + 4 * lc;
  float* o = reinterpret_cast<float*>(out);
#pragma unroll
  for (int it = 0; it < 8; ++it) {
    const int r = it * 4 + lr;
    if (row0 + r < M && col < N)
      *reinterpret_cast<float4*>(o + static_cast<int64_t>(row0 + r) * e.ldo + col) = stg[r * 8 + (lc ^ (r & 7))];
  }
  __syncwarp();
}

// Epilogue of one 128 x BN accumulator: this thread owns tile row `row` and handles
// accumulator columns [cb, ce) (gated: output columns [cb, ce) of the BN / 2 the tile
// produces), reading the accumulator through `src`.  `part` (0 or 1) is the column half
// the thread covers, `halves` the number of halves (1 with 4 epilogue warps): a writer of h
// puts its row sums in stat slot 2 n_blk + part.
template <int BN, bool kFastRope, int FEAT, class Src>
__device__ __forceinline__ void epilogue_tile(const TcArgs& a, void* out, int row, int n_blk,
                                              const Src& src, int cb, int ce, int part, int halves,
                                              float4* stg) {
  constexpr int kBN = BN;
  constexpr bool kH16 = FEAT == kFeatH16;
  // compile-time pruning of paths a feature set never takes (gemm_plan enforces it): a
  // folded-norm GEMM has no residual (DELTA) epilogue, a residual writer is DELTA or F32
  constexpr bool kNormFeat = FEAT == kFeatRms || FEAT == kFeatLn;  // (and LayerNorm: no RoPE)
  const EpiParams& e = a.epi;
  const bool row_ok = row < a.M;
  const RowNorm rn = row_norm<FEAT>(e, row, row_ok);
  float x[16], y[16];
  if (!kH16 && a.gated) {
    const int n0 = n_blk * (kBN / 2);
    if constexpr (!kFastRope) {
      if (stg != nullptr) {  // 32 output columns (two 16-column groups) per staged store
#pragma unroll 1
        for (int c = cb; c < ce; c += 32) {
          if (n0 + c >= a.N) break;
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            const int cc = c + 16 * half;
            src.load2(cc, kBN / 2 + cc, x, y);
            apply_norm16<FEAT>(e, rn, n0 + cc, x);
            apply_norm16<FEAT>(e, rn, a.N + n0 + cc, y);
#pragma unroll
            for (int i = 0; i < 16; ++i) x[i] = e.act ? x[i] * gelu_erf_f(y[i]) : silu_f(x[i]) * y[i];
            stage_put16_f16(stg, half, x);
          }
          stage_flush_f16(e, out, row - (threadIdx.x & 31), a.M, a.N, n0 + c, stg);
        }
        return;
      }
    }
    for (int c = cb; c < ce; c += 16) {
      if (n0 + c >= a.N) break;
      src.load2(c, kBN / 2 + c, x, y);
      apply_norm16<FEAT>(e, rn, n0 + c, x);
      apply_norm16<FEAT>(e, rn, a.N + n0 + c, y);
#pragma unroll
      for (int i = 0; i < 16; ++i) x[i] = e.act ? x[i] * gelu_erf_f(y[i]) : silu_f(x[i]) * y[i];
      if (row_ok) {
        if (n0 + c < a.N) epi_store8(e, out, row, n0 + c, x);
        if (n0 + c + 8 < a.N) epi_store8(e, out, row, n0 + c + 8, x + 8);
      }
    }
    return;
  }
  const int n0 = n_blk * kBN;
  if (!kH16 && FEAT != kFeatLn && e.kind == SGD_EPI_ROPE && kFastRope) {
    // every head of the tile shares the row's position, so each 16-wide chunk of the cos /
    // sin tables is read once for all of them and the next chunk is fetched ahead (the
    // 4-epilogue-warp kernel, which has the registers for it)
    const int dh = e.d_head, hd = dh >> 1;
    const int pos = row_ok ? row % e.rope_tokens : 0;
    const float4* cs4 = reinterpret_cast<const float4*>(e.rope_cos + static_cast<int64_t>(pos) * hd);
    const float4* sn4 = reinterpret_cast<const float4*>(e.rope_sin + static_cast<int64_t>(pos) * hd);
    const bool any_rot = row_ok && (n0 + cb) < e.rope_cols;
    float4 cn[4], sn[4];
    if (any_rot) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        cn[i] = cs4[i];
        sn[i] = sn4[i];
      }
    }
    for (int j = 0; j < hd; j += 16) {
      float cc[16], ss[16];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        cc[4 * i] = cn[i].x; cc[4 * i + 1] = cn[i].y; cc[4 * i + 2] = cn[i].z; cc[4 * i + 3] = cn[i].w;
        ss[4 * i] = sn[i].x; ss[4 * i + 1] = sn[i].y; ss[4 * i + 2] = sn[i].z; ss[4 * i + 3] = sn[i].w;
      }
      if (any_rot && j + 16 < hd) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          cn[i] = cs4[(j + 16) / 4 + i];
          sn[i] = sn4[(j + 16) / 4 + i];
        }
      }
      for (int hb = cb; hb < ce; hb += dh) {
        if (n0 + hb >= a.N) break;
        const bool rot = (n0 + hb) < e.rope_cols;
        src.load2(hb + j, hb + hd + j, x, y);
        apply_norm16<FEAT>(e, rn, n0 + hb + j, x);
        apply_norm16<FEAT>(e, rn, n0 + hb + hd + j, y);
        if (rot && row_ok) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float a1 = x[i], a2 = y[i];
            x[i] = a1 * cc[i] - a2 * ss[i];
            y[i] = a2 * cc[i] + a1 * ss[i];
          }
        }
        if (row_ok) {
          const int c1 = n0 + hb + j, c2 = c1 + hd;
          epi_store8(e, out, row, c1, x);
          epi_store8(e, out, row, c1 + 8, x + 8);
          epi_store8(e, out, row, c2, y);
          epi_store8(e, out, row, c2 + 8, y + 8);
        }
      }
    }
    return;
  }
  if (!kH16 && FEAT != kFeatLn && e.kind == SGD_EPI_ROPE && !kFastRope) {
    const int dh = e.d_head, hd = dh >> 1;
    const int pos = row_ok ? row % e.rope_tokens : 0;
    for (int hb = cb; hb < ce; hb += dh) {
      if (n0 + hb >= a.N) break;
      const bool rot = (n0 + hb) < e.rope_cols;
      for (int j = 0; j < hd; j += 16) {
        src.load2(hb + j, hb + hd + j, x, y);
        apply_norm16<FEAT>(e, rn, n0 + hb + j, x);
        apply_norm16<FEAT>(e, rn, n0 + hb + hd + j, y);
        if (rot && row_ok) {
          const float* cs = e.rope_cos + static_cast<int64_t>(pos) * hd + j;
          const float* sn = e.rope_sin + static_cast<int64_t>(pos) * hd + j;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float c_ = cs[i], s_ = sn[i];
            const float a1 = x[i], a2 = y[i];
            x[i] = a1 * c_ - a2 * s_;
            y[i] = a2 * c_ + a1 * s_;
          }
        }
        if (row_ok) {
          const int c1 = n0 + hb + j, c2 = c1 + hd;
          epi_store8(e, out, row, c1, x);
          epi_store8(e, out, row, c1 + 8, x + 8);
          epi_store8(e, out, row, c2, y);
          epi_store8(e, out, row, c2 + 8, y + 8);
        }
      }
    }
    return;
  }
  if (!kNormFeat && e.kind == SGD_EPI_DELTA) {
    if constexpr (!kH16 && !kFastRope) {  // 8-warp kernels (the 4-warp RoPE kernel has no registers to spare)
      if (stg != nullptr) {
        delta_staged(a, row, n0, src, cb, ce, stg);
        return;
      }
    }
    // residual update: the chunk's h (and gate) loads are issued together, ahead of the
    // accumulator reads, instead of one dependent load per 8 columns
    // the residual writer (kFeatH16) serves folded-norm models, which have no AdaLN gate
    const float* grow =
        (!kH16 && e.gate) ? e.gate + static_cast<int64_t>(row_ok ? row / e.rows_per_batch : 0) * e.ld_gate + n0
                          : nullptr;
    float* hrow = e.h + static_cast<int64_t>(row) * e.ldh + n0;
    float st_ss = 0.f, st_s1 = 0.f;
    for (int c = cb; c < ce; c += 32) {
      if (n0 + c >= a.N) break;
      // unconditional loads (a predicated load here makes the compiler spill): columns past
      // N repeat the row's last four, which are read but never used
      float4 hv[8], gv[8];
      const int hr = row_ok ? 0 : -row;  // rows past M read row 0 instead
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int col = min(c + 4 * q, a.N - n0 - 4);
        hv[q] = *reinterpret_cast<const float4*>(hrow + static_cast<int64_t>(hr) * e.ldh + col);
        if constexpr (!kH16)
          gv[q] = grow ? *reinterpret_cast<const float4*>(grow + col) : make_float4(1.f, 1.f, 1.f, 1.f);
      }
      src.load2(c, c + 16, x, y);
      if (row_ok) {
#pragma unroll
        for (int g = 0; g < 4; ++g) {
          if (n0 + c + 8 * g >= a.N) continue;
          float* v = g < 2 ? x + 8 * g : y + 8 * (g - 2);  // constant once unrolled
          if (!kH16 && grow) {
            v[0] *= gv[2 * g].x; v[1] *= gv[2 * g].y; v[2] *= gv[2 * g].z; v[3] *= gv[2 * g].w;
            v[4] *= gv[2 * g + 1].x; v[5] *= gv[2 * g + 1].y; v[6] *= gv[2 * g + 1].z; v[7] *= gv[2 * g + 1].w;
          }
          float4 h0 = hv[2 * g], h1 = hv[2 * g + 1];
          h0.x += v[0]; h0.y += v[1]; h0.z += v[2]; h0.w += v[3];
          h1.x += v[4]; h1.y += v[5]; h1.z += v[6]; h1.w += v[7];
          float4* hp = reinterpret_cast<float4*>(hrow + c + 8 * g);
          hp[0] = h0;
          hp[1] = h1;
          if (e.cache) store8_f16(e.cache, e.ld_cache, row, n0 + c + 8 * g, v);
          if constexpr (kH16) {
            const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
            emit_h8(e, e.ldh, row, n0 + c + 8 * g, hv, st_ss, st_s1);
          }
        }
      }
    }
    if constexpr (kH16) {
      if (row_ok) {
        emit_stats(e, row, 2 * n_blk + part, st_ss, st_s1);
        if (halves == 1) emit_stats(e, row, 2 * n_blk + 1, 0.f, 0.f);
      }
    }
    return;
  }
  if constexpr (!kH16 && !kFastRope) {
    if (stg != nullptr && (e.kind == SGD_EPI_F16 || e.kind == SGD_EPI_GELU || e.kind == SGD_EPI_F32)) {
#pragma unroll 1
      for (int c = cb; c < ce; c += 32) {
        if (n0 + c >= a.N) break;
        src.load2(c, c + 16, x, y);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          float* v = half ? y : x;
          apply_norm16<FEAT>(e, rn, n0 + c + 16 * half, v);
          if (e.kind == SGD_EPI_GELU) {
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = e.act ? gelu_erf_f(v[i]) : gelu_tanh_f(v[i]);
          }
          if (e.kind == SGD_EPI_F32)
            stage_put16_f32(stg, half, v);
          else
            stage_put16_f16(stg, half, v);
        }
        if (e.kind == SGD_EPI_F32)
          stage_flush_f32(e, out, row - (threadIdx.x & 31), a.M, a.N, n0 + c, stg);
        else
          stage_flush_f16(e, out, row - (threadIdx.x & 31), a.M, a.N, n0 + c, stg);
      }
      return;
    }
  }
  float st_ss = 0.f, st_s1 = 0.f;
  for (int c = cb; c < ce; c += 32) {
    if (n0 + c >= a.N) break;
    src.load2(c, c + 16, x, y);
    // the first 16 columns are normalised and stored before the second 16 are touched (the
    // LayerNorm column vectors of one half at a time)
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      float* v = half ? y : x;
      const int c0 = n0 + c + 16 * half;
      apply_norm16<FEAT>(e, rn, c0, v);
      if (row_ok) {
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          if (c0 + 8 * q < a.N) {
            epi_store8(e, out, row, c0 + 8 * q, v + 8 * q);
            if constexpr (kH16) emit_h8(e, e.ldo, row, c0 + 8 * q, v + 8 * q, st_ss, st_s1);
          }
        }
      }
    }
  }
  if constexpr (kH16) {
    if (row_ok) {
      emit_stats(e, row, 2 * n_blk + part, st_ss, st_s1);
      if (halves == 1) emit_stats(e, row, 2 * n_blk + 1, 0.f, 0.f);
    }
  }
}

// Wait on a barrier with the whole warp: lane 0 polls, the verdict is broadcast so
// that the warp stays converged for the .sync.aligned tcgen05 instructions.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          int* status, int code) {
  int ok = 0;
  if (lane_id() == 0) ok = mbar_wait(bar, parity, abort_flag, status, code) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  return ok != 0;
}

// Bounded wait that ignores the abort flag (used while draining after an abort).
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitTimeoutNs) break;
  }
}

// Named barrier 1 over the epilogue warps, returning the AND of `v` over them.
__device__ __forceinline__ bool epi_bar_and(bool v, int nthreads) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, %2, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "r"(nthreads)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ void epi_bar(int nthreads) {
  asm volatile("bar.sync 1, %0;" ::"r"(nthreads) : "memory");
}

// Output tile of linear tile index t.  group_m = 0: M-fastest (m = t % num_m).  group_m = G:
// the row-blocks form groups of G; a group's tiles come one after another, column by column
// (G row-blocks of one column, then the next column), and every other group walks its
// columns backwards.  A wave of CTAs then covers about G row-blocks by (CTAs / G) columns,
// so its A rows are shared by all of its columns, and consecutive groups start on the
// columns the previous one ended on (still in L2).
__device__ __forceinline__ void tile_coords(const TcArgs& a, int t, int& m_blk, int& n_blk) {
  if (a.group_m <= 0) {
    m_blk = t % a.num_m;
    n_blk = t / a.num_m;
    return;
  }
  const int per_group = a.group_m * a.num_n;
  const int g = t / per_group, w = t - g * per_group;
  const int gm = min(a.group_m, a.num_m - g * a.group_m);  // row-blocks in this (last) group
  const int col = w / gm;
  m_blk = g * a.group_m + (w - col * gm);
  n_blk = (g & 1) ? a.num_n - 1 - col : col;
}

// Stream-K split of the K iterations of tiles [0, sk_tiles): CTA c < sk_ctas owns the
// contiguous iterations [start(c), start(c + 1)) of the sk_tiles * num_k iteration space,
// start(c) = floor(c * total / sk_ctas); every CTA owns at least one iteration (the host
// keeps sk_ctas <= total).  The CTA owning iteration i is the largest c with start(c) <= i.
__device__ __forceinline__ int sk_start(int c, int total, int ctas) {
  return static_cast<int>(static_cast<int64_t>(c) * total / ctas);
}
__device__ __forceinline__ int sk_owner(int i, int total, int ctas) {
  return static_cast<int>((static_cast<int64_t>(i + 1) * ctas - 1) / total);
}

// The work of one CTA: first its stream-K segments (tiles t_sk0 .., K iterations clipped to
// [sk_s, sk_e)), then the data-parallel tiles sk_tiles + unit0 + d * unit_step, full K.
struct CtaWork {
  int sk_s, sk_e, t_sk0, n_sk;
  int unit0, unit_step, n_units;
};

__device__ __forceinline__ CtaWork cta_work(const TcArgs& a, int num_tiles, int unit0, int unit_step) {
  CtaWork w;
  w.unit0 = unit0;
  w.unit_step = unit_step;
  w.sk_s = w.sk_e = w.t_sk0 = w.n_sk = 0;
  if (a.sk_tiles > 0 && static_cast<int>(blockIdx.x) < a.sk_ctas) {
    const int total = a.sk_tiles * a.num_k;
    w.sk_s = sk_start(blockIdx.x, total, a.sk_ctas);
    w.sk_e = sk_start(blockIdx.x + 1, total, a.sk_ctas);
    w.t_sk0 = w.sk_s / a.num_k;
    w.n_sk = (w.sk_e - 1) / a.num_k - w.t_sk0 + 1;
  }
  const int dp = num_tiles - a.sk_tiles;
  const int n_dp = unit0 < dp ? (dp - unit0 + unit_step - 1) / unit_step : 0;
  w.n_units = w.n_sk + n_dp;
  return w;
}

__device__ __forceinline__ void unit_at(const TcArgs& a, const CtaWork& w, int u, int& tile, int& k0,
                                        int& k1) {
  if (u < w.n_sk) {
    tile = w.t_sk0 + u;
    const int base = tile * a.num_k;
    k0 = max(w.sk_s - base, 0);
    k1 = min(w.sk_e - base, a.num_k);
  } else {
    tile = a.sk_tiles + w.unit0 + (u - w.n_sk) * w.unit_step;
    k0 = 0;
    k1 = a.num_k;
  }
}

// Residual writer with finalisation (EpiParams::stat_cnt): after the epilogue of a tile, every
// epilogue thread takes part (also after an expired wait, so that all leave together; returns
// false then).  The tile's partial sums are published (fence), one thread draws a ticket for
// the tile's row block, and the CTA holding the last ticket sums the block's slots per row
// (one thread per row) into stat_final and resets the counter.
template <int kEpiThreads>
__device__ __forceinline__ bool finalize_row_stats(const TcArgs& a, bool ok, int m_blk, int row, bool row_owner,
                                                   volatile int* fin_flag) {
  const EpiParams& e = a.epi;
  __threadfence();
  if (!epi_bar_and(ok, kEpiThreads)) return false;
  if (threadIdx.x == 64) *fin_flag = atomicAdd(&e.stat_cnt[m_blk], 1) == a.num_n - 1 ? 1 : 0;
  epi_bar(kEpiThreads);
  if (*fin_flag != 0) {
    __threadfence();
    if (row_owner && row < a.M) {
      const int slots = 2 * a.num_n;
      const int64_t ld = e.stat_out_ld;
      e.stat_final[row] = sum_slots(e.stat_out + row, ld, slots);
      e.stat_final[static_cast<int64_t>(kStatSlots) * ld + row] =
          sum_slots(e.stat_out + static_cast<int64_t>(kStatSlots) * ld + row, ld, slots);
    }
    if (threadIdx.x == 64) e.stat_cnt[m_blk] = 0;
  }
  // fin_flag is rewritten (next tile) only after every epilogue thread has read it: each
  // reads it before it reaches the next tile's first barrier
  return true;
}

// Stream-K (sk_tiles > 0): the K iterations of the first sk_tiles tiles are
// spread evenly over sk_ctas CTAs (at most kMaxSeg per tile), so that the tiles left over
// after the last full wave do not leave most SMs idle.  A CTA whose segment does not cover
// a tile's whole K range stores its raw accumulator in its workspace slot, then draws a
// ticket from the tile's counter; the CTA that draws the last ticket sums the slots in
// order, runs the epilogue and puts the counter back to zero.  No CTA ever waits for
// another.
template <int BK, int BN, int EPIW, int FEAT>
__global__ void __launch_bounds__(TileCfg<BK, BN, EPIW>::kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ TcArgs a) {
  using C = TileCfg<BK, BN, EPIW>;
  constexpr int kBK = C::kBK, kStages = C::kStages, kTileA = C::kTileA;
  constexpr int kTileBHalf = C::kTileBHalf, kStageBytes = C::kStageBytes;
  constexpr int kBN = C::kBN, kTmemCols = C::kTmemCols, kEpiWarps = C::kEpiWarps;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* tiles = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(tiles + kStages * kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_slot + 2);
  volatile int* fin_flag = reinterpret_cast<volatile int*>(tmem_slot + 3);
  // this epilogue warp's staging buffer (after the 256-byte barrier block), if the tile has one
  float4* stg = nullptr;
  if constexpr (C::kStaging > 0) {
    if (threadIdx.x >= 64)
      stg = reinterpret_cast<float4*>(tiles + kStages * kStageBytes + 256) + ((threadIdx.x >> 5) - 2) * 256;
  }

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&a.tmap_a);
    tma_prefetch_desc(&a.tmap_b);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait_and_trigger();  // the prologue above touched only shared memory and TMEM
  const uint32_t tmem_base = *tmem_slot;
  const int num_mu = a.num_m;
  const int num_tiles = num_mu * a.num_n;
  const CtaWork w = cta_work(a, num_tiles, blockIdx.x, gridDim.x);

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      for (int u = 0; u < w.n_units; ++u) {
        int tile, k0, k1;
        unit_at(a, w, u, tile, k0, k1);
        int m_blk, n_blk;
        tile_coords(a, tile, m_blk, n_blk);
        const int rb0 = a.gated ? n_blk * 128 : n_blk * kBN;
        const int rb1 = a.gated ? a.N + n_blk * 128 : rb0 + 128;  // BN = 256 only
        bool ok = true;
        for (int kb = k0; kb < k1; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status, 1)) {
            ok = false;
            break;
          }
          uint8_t* st = tiles + s * kStageBytes;
          mbar_arrive_expect_tx(&full[s], kStageBytes);
          tma_load_2d(st, &a.tmap_a, &full[s], kb * kBK, m_blk * kBM);
          tma_load_2d(st + kTileA, &a.tmap_b, &full[s], kb * kBK, rb0);
          if (kBN == 256) tma_load_2d(st + kTileA + kTileBHalf, &a.tmap_b, &full[s], kb * kBK, rb1);
        }
        if (!ok) break;
      }
      if (*abort_flag) {
        // wait for the loads still in flight (the latest issue of each stage)
        for (int i = (it > kStages ? it - kStages : 0); i < it; ++i)
          drain_wait(&full[i % kStages], (i / kStages) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_f16(kBM, kBN);
      int it = 0;
      bool ok = true;
      for (int u = 0; u < w.n_units && ok; ++u) {
        int tile, k0, k1;
        unit_at(a, w, u, tile, k0, k1);
        const int acc = u & 1;
        const uint32_t aph = (u >> 1) & 1;
        if (!mbar_wait(&tempty[acc], aph ^ 1u, abort_flag, a.status, 2)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * kBN;
        for (int kb = k0; kb < k1; ++kb, ++it) {
          const int s = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, a.status, 3)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_u32(tiles + s * kStageBytes);
          const uint32_t b_addr = a_addr + kTileA;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            umma_f16(d_tmem, operand_desc<BK>(a_addr + 32 * k), operand_desc<BK>(b_addr + 32 * k),
                      idesc, (kb != k0 || k != 0) ? 1u : 0u);
          }
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
      }
      // every MMA issued by this thread has finished once `drain` completes
      umma_commit(drain);
      drain_wait(drain, 0);
    }
  } else {
    const int q = warp & 3;
    constexpr int kEpiThreads = 32 * kEpiWarps;
    // column range of this warp: all of the tile (4 epilogue warps) or one half (8)
    // (8 warps: the first half rounded up to a multiple of 32 columns, e.g. 128 + 96 at BN 224)
    constexpr int kSplit = ((kBN / 2 + 31) / 32) * 32, kSplitGated = ((kBN / 4 + 31) / 32) * 32;
    const int span = a.gated ? kBN / 2 : kBN;
    const int part = kEpiWarps == 8 ? ((warp - 2) >> 2) : 0;
    const int split = a.gated ? kSplitGated : kSplit;
    const int cb = kEpiWarps == 8 ? part * split : 0;
    const int ce = kEpiWarps == 8 ? (part ? span : split) : span;
    // accumulator columns this warp stores for a stream-K partial
    const int pb = kEpiWarps == 8 ? part * kSplit : 0;
    const int pe = kEpiWarps == 8 ? (part ? kBN : kSplit) : kBN;
    const int total = a.sk_tiles * a.num_k;
    void* out = a.epi.out_slot ? *a.epi.out_slot : a.epi.out;
    for (int u = 0; u < w.n_units; ++u) {
      int tile, k0, k1;
      unit_at(a, w, u, tile, k0, k1);
      int m_blk, n_blk;
      tile_coords(a, tile, m_blk, n_blk);
      const int acc = u & 1;
      const uint32_t aph = (u >> 1) & 1;
      const int row = m_blk * kBM + q * 32 + lane;
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + acc * kBN;
      if (u >= w.n_sk) {  // data-parallel tile
        prefetch_h_row(a.epi, row, a.M, a.N, n_blk * kBN, cb, ce);
        if (FEAT == kFeatH16 && a.epi.stat_cnt) {  // every epilogue thread reaches the barriers
          const bool ok = warp_wait(&tfull[acc], aph, abort_flag, a.status, 4);
          if (ok) {
            tc_fence_after();
            epilogue_tile<kBN, kEpiWarps == 4, FEAT>(a, out, row, n_blk, TmemSrc{tbase, a.epi.alpha}, cb, ce,
                                                     part, kEpiWarps == 8 ? 2 : 1, stg);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
          }
          if (!finalize_row_stats<kEpiThreads>(a, ok, m_blk, row, part == 0, fin_flag)) break;
          continue;
        }
        if (!warp_wait(&tfull[acc], aph, abort_flag, a.status, 4)) break;
        tc_fence_after();
        epilogue_tile<kBN, kEpiWarps == 4, FEAT>(a, out, row, n_blk, TmemSrc{tbase, a.epi.alpha}, cb, ce, part,
                                           kEpiWarps == 8 ? 2 : 1, stg);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        continue;
      }
      // stream-K unit: every epilogue warp reaches each barrier below, also after an
      // expired wait, so that they leave the loop together
      const bool ok = warp_wait(&tfull[acc], aph, abort_flag, a.status, 4);
      if (k0 == 0 && k1 == a.num_k) {  // the whole K range of the tile lies in this CTA's share
        if (ok) {
          tc_fence_after();
          epilogue_tile<kBN, kEpiWarps == 4, FEAT>(a, out, row, n_blk, TmemSrc{tbase, a.epi.alpha}, cb, ce, part,
                                           kEpiWarps == 8 ? 2 : 1, stg);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&tempty[acc]);
        }
        if (FEAT == kFeatH16 && a.epi.stat_cnt) {
          if (!finalize_row_stats<kEpiThreads>(a, ok, m_blk, row, part == 0, fin_flag)) break;
          continue;
        }
        if (!epi_bar_and(ok, kEpiThreads)) break;
        continue;
      }
      // partial: store it, then draw a ticket; the CTA that draws the last one has every
      // other partial in the workspace already and finishes the tile.  No CTA waits.
      const int first = sk_owner(tile * a.num_k, total, a.sk_ctas);
      const int nseg = sk_owner(tile * a.num_k + a.num_k - 1, total, a.sk_ctas) - first + 1;
      float* slot0 = a.ws + static_cast<size_t>(tile) * a.max_seg * (kBM * kBN);
      if (ok) {
        tc_fence_after();
        store_partial<kBN>(slot0 + static_cast<size_t>(blockIdx.x - first) * (kBM * kBN), q * 32 + lane,
                           tbase, pb, pe);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        __threadfence();
      }
      if (!epi_bar_and(ok, kEpiThreads)) break;
      // last_flag is rewritten (next stream-K unit) only after every epilogue thread has
      // read it, since each reads it before reaching the next epi_bar_and
      if (threadIdx.x == 64) {
        __threadfence();
        *last_flag = atomicAdd(&a.sk_cnt[tile], 1) == nseg - 1 ? 1 : 0;
      }
      epi_bar(kEpiThreads);
      if (*last_flag != 0) {
        __threadfence();
        epilogue_tile<kBN, kEpiWarps == 4, FEAT>(a, out, row, n_blk, WsSrc<kBN>{slot0, nseg, q * 32 + lane, a.epi.alpha},
                                           cb, ce, part, kEpiWarps == 8 ? 2 : 1, stg);
        if (threadIdx.x == 64) a.sk_cnt[tile] = 0;
      }
      // the CTA that finished the tile (last_flag is CTA-uniform) draws its row block's ticket
      if (FEAT == kFeatH16 && a.epi.stat_cnt && *last_flag != 0) {
        if (!finalize_row_stats<kEpiThreads>(a, true, m_blk, row, part == 0, fin_flag)) break;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}


template <int BK, int BN, int EPIW, int FEAT>
cudaError_t launch_tc(const GemmPlan& p, const TcArgs& a, cudaStream_t s) {
  constexpr int kSmemBytes = TileCfg<BK, BN, EPIW>::kSmemBytes;
  constexpr int kThreads = TileCfg<BK, BN, EPIW>::kThreads;
  static bool attr_done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !attr_done[dev]) {
    cudaError_t err = cudaFuncSetAttribute(gemm_tc_kernel<BK, BN, EPIW, FEAT>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (err != cudaSuccess) return err;
    attr_done[dev] = true;
  }
  return launch_k(gemm_tc_kernel<BK, BN, EPIW, FEAT>, dim3(p.grid), dim3(kThreads), kSmemBytes, s, a);
}


}  // namespace gk
}  // namespace sgd
