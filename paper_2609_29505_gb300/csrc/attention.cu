// Non-causal multi-head attention O = softmax(Q K^T / sqrt(d_h)) V, flash style.
//
// Used inside every active self-attention and cross-attention branch (Algorithm 2:
// an active unit evaluates F_l(h_{l-1,s}; c_s)); frozen units never launch it.
//
// Three kernels:
//   attn_pp_kernel (d_h 64, 128; the default): tcgen05 with two query tiles per CTA and two
//     alternating softmax warpgroups, P in TMEM; described above the kernel.
//   attn_tc_kernel (d_h 64, 128): tcgen05.  One CTA = 128 queries of one (sample, head),
//     keys in tiles of 128.  Warp 0 loads Q once and K/V tiles through a 2-stage TMA ring;
//     warp 1 issues S = Q K^T into one of two TMEM S buffers and O += P V into a TMEM O
//     accumulator (V read as an MN-major operand straight from its row-major tile);
//     warps 2-5 (one query row per thread) read S from TMEM, run the online softmax in
//     fp32 and write P (fp16) into a 128-byte-swizzled shared tile for the next MMA.  O
//     is rescaled only when a row maximum grows by more than 2^8 (P <= 256 otherwise),
//     which keeps the result exact while avoiding most TMEM round trips.
//   attn_kernel (any of 64, 72, 128): mma.sync, described below; used for d_h = 72.
//
// mma.sync kernel: one CTA = 64 query rows of one (sample, head), 4 warps x 16 rows.  K/V tiles of
// 64 keys stream through a double-buffered cp.async ring; S = Q K^T and O += P V run
// on mma.sync m16n8k16 (fp16 in, fp32 accumulate) with an online softmax in
// registers (exp2 with the scale folded in).  Q, K, V, P and O are fp16 (m16n8k16
// f16 x f16 -> f32).  Keys beyond n_kv are masked and their
// shared-memory rows zero-filled; head dims 72 are padded to 80 in shared memory.
#include <cstring>

#include "common.cuh"
#include "kernels.h"

namespace sgd {

namespace {

constexpr int kBQ = 64;
constexpr int kBKV = 64;
constexpr int kWarps = 4;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t s = smem_u32(smem);
  const int sz = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(gmem), "r"(sz)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ void mma_f16_16816(float* c, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// DP: padded head dim in shared memory (multiple of 16); DH: real head dim.
template <int DH, int DP>
__global__ void __launch_bounds__(kWarps * 32) attn_kernel(const AttnParams p) {
  constexpr int kPitch = DP + 8;           // elements per shared row (bank-conflict free)
  constexpr int kChunks = DH / 8;          // 16-byte chunks of real data per row
  constexpr int kPadChunks = DP / 8;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  f16* sQ = reinterpret_cast<f16*>(smem_raw);
  f16* sK = sQ + kBQ * kPitch;            // [2][kBKV][kPitch]
  f16* sV = sK + 2 * kBKV * kPitch;       // [2][kBKV][kPitch]

  pdl_wait_and_trigger();
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int q0 = blockIdx.x * kBQ;
  const int bh = blockIdx.y;
  const int b = bh / p.n_heads, h = bh % p.n_heads;
  const int hs = p.head_stride > 0 ? p.head_stride : DH;  // input columns between heads
  const f16* qbase = p.q + (static_cast<int64_t>(b) * p.n_q) * p.ldq + h * hs;
  const f16* kbase = p.k + (static_cast<int64_t>(b) * p.n_kv) * p.ldkv + h * hs;
  const f16* vbase = p.v + (static_cast<int64_t>(b) * p.n_kv) * p.ldkv + h * hs;

  // Q tile
  for (int i = tid; i < kBQ * kPadChunks; i += kWarps * 32) {
    const int r = i / kPadChunks, c = i % kPadChunks;
    const bool ok = (q0 + r) < p.n_q && c < kChunks;
    const f16* src = ok ? qbase + static_cast<int64_t>(q0 + r) * p.ldq + c * 8 : p.q;
    cp_async16(sQ + r * kPitch + c * 8, src, ok);
  }
  auto load_kv = [&](int tile, int buf) {
    const int k0 = tile * kBKV;
    f16* dk = sK + buf * kBKV * kPitch;
    f16* dv = sV + buf * kBKV * kPitch;
    for (int i = tid; i < kBKV * kPadChunks; i += kWarps * 32) {
      const int r = i / kPadChunks, c = i % kPadChunks;
      const bool ok = (k0 + r) < p.n_kv && c < kChunks;
      const int64_t off = static_cast<int64_t>(k0 + r) * p.ldkv + c * 8;
      cp_async16(dk + r * kPitch + c * 8, ok ? kbase + off : p.k, ok);
      cp_async16(dv + r * kPitch + c * 8, ok ? vbase + off : p.v, ok);
    }
  };
  const int n_tiles = (p.n_kv + kBKV - 1) / kBKV;
  load_kv(0, 0);
  cp_async_commit();

  constexpr int KS = DP / 16;   // k-steps over the head dim
  constexpr int NO = DP / 8;    // output n-tiles
  uint32_t qf[KS][4];
  float o[NO][4];
#pragma unroll
  for (int i = 0; i < NO; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};
  const float sl2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));  // log2(e)/sqrt(d_h)
  const int g = lane >> 2, t4 = lane & 3;

  for (int tile = 0; tile < n_tiles; ++tile) {
    const int buf = tile & 1;
    if (tile + 1 < n_tiles) {
      load_kv(tile + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (tile == 0) {
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int r = warp * 16 + (lane & 15);
        const int c = ks * 16 + (lane >> 4) * 8;
        ldmatrix_x4(qf[ks], sQ + r * kPitch + c);
      }
    }
    const f16* tk = sK + buf * kBKV * kPitch;
    const f16* tv = sV + buf * kBKV * kPitch;
    // S = Q K^T : 16 x 64 per warp
    float s[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t kb[4];
        const int r = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = ks * 16 + ((lane >> 3) & 1) * 8;
        ldmatrix_x4(kb, tk + r * kPitch + c);
        mma_f16_16816(s[2 * np], qf[ks], kb);
        mma_f16_16816(s[2 * np + 1], qf[ks], kb + 2);
      }
    }
    // mask keys beyond n_kv
    const int kbase_idx = tile * kBKV;
    if (kbase_idx + kBKV > p.n_kv) {
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        const int j = kbase_idx + nt * 8 + 2 * t4;
        if (j >= p.n_kv) { s[nt][0] = -INFINITY; s[nt][2] = -INFINITY; }
        if (j + 1 >= p.n_kv) { s[nt][1] = -INFINITY; s[nt][3] = -INFINITY; }
      }
    }
    // online softmax (rows g and g + 8 of this warp's 16)
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      mx[0] = fmaxf(mx[0], fmaxf(s[nt][0], s[nt][1]));
      mx[1] = fmaxf(mx[1], fmaxf(s[nt][2], s[nt][3]));
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
    }
    float corr[2], mnew[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mnew[r] = fmaxf(m_r[r], mx[r]);
      corr[r] = exp2f((m_r[r] - mnew[r]) * sl2);
      m_r[r] = mnew[r];
    }
    float rs[2] = {0.f, 0.f};
    uint32_t pf[4][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = exp2f((s[nt][0] - mnew[0]) * sl2);
      const float p1 = exp2f((s[nt][1] - mnew[0]) * sl2);
      const float p2 = exp2f((s[nt][2] - mnew[1]) * sl2);
      const float p3 = exp2f((s[nt][3] - mnew[1]) * sl2);
      rs[0] += p0 + p1;
      rs[1] += p2 + p3;
      const int kk = nt >> 1, hi = nt & 1;
      pf[kk][hi * 2 + 0] = pack_f16x2(p0, p1);
      pf[kk][hi * 2 + 1] = pack_f16x2(p2, p3);
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 1);
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 2);
      l_r[r] = l_r[r] * corr[r] + rs[r];
    }
#pragma unroll
    for (int i = 0; i < NO; ++i) {
      o[i][0] *= corr[0]; o[i][1] *= corr[0];
      o[i][2] *= corr[1]; o[i][3] *= corr[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      // A fragment order: a0 (row g, k 0-7), a1 (row g+8, k 0-7), a2 (row g, k 8-15), a3
      uint32_t a[4] = {pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3]};
#pragma unroll
      for (int np = 0; np < NO / 2; ++np) {
        uint32_t vb[4];
        const int r = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int c = np * 16 + (lane >> 4) * 8;
        ldmatrix_x4_trans(vb, tv + r * kPitch + c);
        mma_f16_16816(o[2 * np], a, vb);
        mma_f16_16816(o[2 * np + 1], a, vb + 2);
      }
    }
    __syncthreads();
  }
  // normalise and store
  const float inv0 = 1.f / l_r[0], inv1 = 1.f / l_r[1];
  const int row0 = q0 + warp * 16 + g, row1 = row0 + 8;
  f16* ob = p.o + (static_cast<int64_t>(b) * p.n_q) * p.ldo + h * DH;
#pragma unroll
  for (int nt = 0; nt < NO; ++nt) {
    const int c = nt * 8 + 2 * t4;
    if (c < DH) {
      if (row0 < p.n_q)
        *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(row0) * p.ldo + c) =
            pack_f16x2(o[nt][0] * inv0, o[nt][1] * inv0);
      if (row1 < p.n_q)
        *reinterpret_cast<uint32_t*>(ob + static_cast<int64_t>(row1) * p.ldo + c) =
            pack_f16x2(o[nt][2] * inv1, o[nt][3] * inv1);
    }
  }
}

// ----------------------------------------------------------------------------
// tcgen05 flash attention
// ----------------------------------------------------------------------------

constexpr int kTcThreads = 192;
constexpr int kTcBQ = 128;
constexpr int kTcBK = 128;
constexpr int kAtom = 128 * 64 * 2;  // 128 rows x 64 fp16: one 128-byte-swizzle column block
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the row max grows by > 2^8

// fp16 pair, round to nearest, no saturation (the callers' values are far below 65504)
__device__ __forceinline__ uint32_t pack_f16x2_rn(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// 2^x with the hardware's approximate base-2 exponential (PTX ex2.approx.ftz.f32); the
// arguments here are <= 8 and results below the fp16 range flush to zero either way.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct AttnTcArgs {
  CUtensorMap tmap_q;
  CUtensorMap tmap_k;
  CUtensorMap tmap_v;
  // d_h = 72 (heads padded to 80 columns in the input): boxes of the last 16 columns
  CUtensorMap tmap_q16;
  CUtensorMap tmap_k16;
  CUtensorMap tmap_v16;
  int head_stride;  // input columns between heads
  f16* o;
  int ldo;
  int n_q, n_kv, n_heads;
  float scale_log2;
  int* status;
};

template <int DH>
struct TcLayout {
  static constexpr int kAtoms = DH / 64;
  static constexpr int kQ = 0;
  static constexpr int kKV = kAtoms * kAtom;           // stage s: K atoms, then V atoms
  static constexpr int kStage = 2 * kAtoms * kAtom;
  static constexpr int kP = kKV + 2 * kStage;          // two P buffers of 128 keys
  static constexpr int kPBuf = 2 * kAtom;
  static constexpr int kBar = kP + 2 * kPBuf;
  static constexpr int kBytes = kBar + 256 + 1024;
  static constexpr uint32_t kTmemS = 0;                // S buffers at columns 0, 128
  static constexpr uint32_t kTmemO = 256;              // O at columns 256 .. 256 + DH
};

__device__ __forceinline__ bool warp_wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                              int* status, int code) {
  int ok = 0;
  if (lane_id() == 0) ok = mbar_wait(bar, parity, abort_flag, status, code) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

__device__ __forceinline__ void drain_bar(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitTimeoutNs) break;
  }
}

template <int DH>
__global__ void __launch_bounds__(kTcThreads, 1) attn_tc_kernel(const __grid_constant__ AttnTcArgs a) {
  using L = TcLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kBar);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = bars + 3;
  uint64_t* s_full = bars + 5;
  uint64_t* s_free = bars + 7;
  uint64_t* p_full = bars + 9;
  uint64_t* o_done = bars + 11;
  uint64_t* drain = bars + 13;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 14);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.n_heads, h = bh % a.n_heads;
  const int nt = (a.n_kv + kTcBK - 1) / kTcBK;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 4);
      mbar_init(&p_full[i], 4);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&a.tmap_q);
    tma_prefetch_desc(&a.tmap_k);
    tma_prefetch_desc(&a.tmap_v);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait_and_trigger();  // the prologue above touched only shared memory and TMEM
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(q_full, L::kAtoms * kAtom);
      for (int at = 0; at < L::kAtoms; ++at)
        tma_load_2d(sm + L::kQ + at * kAtom, &a.tmap_q, q_full, h * a.head_stride + at * 64,
                    b * a.n_q + qt * kTcBQ);
      int j = 0;
      for (; j < nt; ++j) {
        const int s = j & 1;
        if (!mbar_wait(&kv_empty[s], ((j >> 1) & 1) ^ 1u, abort_flag, a.status, 11)) break;
        uint8_t* st = sm + L::kKV + s * L::kStage;
        mbar_arrive_expect_tx(&kv_full[s], 2 * L::kAtoms * kAtom);
        const int row = b * a.n_kv + j * kTcBK;
        for (int at = 0; at < L::kAtoms; ++at) {
          tma_load_2d(st + at * kAtom, &a.tmap_k, &kv_full[s], h * a.head_stride + at * 64, row);
          tma_load_2d(st + (L::kAtoms + at) * kAtom, &a.tmap_v, &kv_full[s], h * a.head_stride + at * 64, row);
        }
      }
      if (*abort_flag) {
        drain_bar(q_full, 0);
        for (int i = (j > 2 ? j - 2 : 0); i < j; ++i) drain_bar(&kv_full[i & 1], (i >> 1) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc_qk = umma_idesc_f16(kTcBQ, kTcBK);
      const uint32_t idesc_pv = umma_idesc_f16_bmn(kTcBQ, DH);
      bool ok = mbar_wait(q_full, 0, abort_flag, a.status, 12);
      auto issue_qk = [&](int j) -> bool {
        const int s = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!mbar_wait(&kv_full[s], ph, abort_flag, a.status, 13)) return false;
        if (!mbar_wait(&s_free[s], ph ^ 1u, abort_flag, a.status, 14)) return false;
        tc_fence_after();
        const uint32_t qa = smem_u32(sm + L::kQ);
        const uint32_t ka = smem_u32(sm + L::kKV + s * L::kStage);
#pragma unroll
        for (int ks = 0; ks < DH / 16; ++ks) {
          const uint32_t off = (ks >> 2) * kAtom + (ks & 3) * 32;
          umma_f16(tmem + L::kTmemS + s * kTcBK, smem_desc_sw128(qa + off), smem_desc_sw128(ka + off),
                   idesc_qk, ks > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[s]);
        return true;
      };
      if (ok) ok = issue_qk(0);
      for (int j = 0; j < nt && ok; ++j) {
        if (j + 1 < nt && !(ok = issue_qk(j + 1))) break;
        const int s = j & 1;
        if (!(ok = mbar_wait(&p_full[s], (j >> 1) & 1, abort_flag, a.status, 15))) break;
        tc_fence_after();
        const uint32_t pa = smem_u32(sm + L::kP + s * L::kPBuf);
        const uint32_t va = smem_u32(sm + L::kKV + s * L::kStage + L::kAtoms * kAtom);
#pragma unroll
        for (int ks = 0; ks < kTcBK / 16; ++ks) {
          const uint64_t ad = smem_desc_sw128(pa + (ks >> 2) * kAtom + (ks & 3) * 32);
          const uint64_t bd = smem_desc_sw128_mn(va + ks * 2048, kAtom, 1024);
          umma_f16(tmem + L::kTmemO, ad, bd, idesc_pv, (j > 0 || ks > 0) ? 1u : 0u);
        }
        umma_commit(&kv_empty[s]);
        umma_commit(&o_done[s]);
      }
      umma_commit(drain);
      drain_bar(drain, 0);
    }
  } else {
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
    float m2 = -INFINITY, l = 0.f;
    bool ok = true;
    uint32_t r[kTcBK];
    for (int j = 0; j < nt; ++j) {
      const int s = j & 1;
      if (!(ok = warp_wait_bar(&s_full[s], (j >> 1) & 1, abort_flag, a.status, 16))) break;
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < kTcBK / 16; ++c) tmem_ld16(tmem + lane_base + L::kTmemS + s * kTcBK + 16 * c, r + 16 * c);
#pragma unroll
      for (int c = 0; c < kTcBK / 16; ++c) tmem_ld_wait16(r + 16 * c);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[s]);
      const int kb = j * kTcBK;
      // scores in log2 units; 8 independent max chains (one softmax warp per SM
      // sub-partition: the reductions are latency-, not throughput-bound)
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = -INFINITY;
      if (kb + kTcBK <= a.n_kv) {
#pragma unroll
        for (int c = 0; c < kTcBK; ++c) {
          const float v = __uint_as_float(r[c]) * a.scale_log2;
          r[c] = __float_as_uint(v);
          mx[c & 7] = fmaxf(mx[c & 7], v);
        }
      } else {
#pragma unroll
        for (int c = 0; c < kTcBK; ++c) {
          const float v = (kb + c < a.n_kv) ? __uint_as_float(r[c]) * a.scale_log2 : -INFINITY;
          r[c] = __float_as_uint(v);
          mx[c & 7] = fmaxf(mx[c & 7], v);
        }
      }
      const float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                             fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      if (j == 0) {
        m2 = mt;
      } else if (__any_sync(0xffffffffu, mt > m2 + kRescaleLog2)) {
        // Warp-uniform branch (the TMEM loads and stores below are .sync.aligned): every
        // lane moves its reference to max(m2, mt), which keeps O / l exact.  O must hold
        // PV_{j-1} complete before it is rescaled.
        if (!(ok = warp_wait_bar(&o_done[(j - 1) & 1], ((j - 1) >> 1) & 1, abort_flag, a.status, 17))) break;
        tc_fence_after();
        const float mnew = fmaxf(m2, mt);
        const float corr = exp2f(m2 - mnew);
        uint32_t o16[16];
#pragma unroll
        for (int c = 0; c < DH / 16; ++c) {
          tmem_ld16(tmem + lane_base + L::kTmemO + 16 * c, o16);
          tmem_ld_wait16(o16);
#pragma unroll
          for (int i = 0; i < 16; ++i) o16[i] = __float_as_uint(__uint_as_float(o16[i]) * corr);
          tmem_st16(tmem + lane_base + L::kTmemO + 16 * c, o16);
        }
        tmem_st_wait();
        tc_fence_before();
        l *= corr;
        m2 = mnew;
      }
      // P buffer s was last read by PV_{j-2}
      if (j >= 2 && !(ok = warp_wait_bar(&o_done[s], ((j - 2) >> 1) & 1, abort_flag, a.status, 18))) break;
      uint8_t* pbuf = sm + L::kP + s * L::kPBuf;
      float ls[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ls[i] = 0.f;
#pragma unroll
      for (int cc = 0; cc < kTcBK / 8; ++cc) {
        float p8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          p8[i] = exp2f(__uint_as_float(r[cc * 8 + i]) - m2);
          ls[i] += p8[i];
        }
        uint8_t* dst = pbuf + (cc >> 3) * kAtom + row * 128 + ((((cc & 7) ^ (row & 7))) << 4);
        *reinterpret_cast<uint4*>(dst) = pack_f16x8(p8);
      }
      l += ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[s]);
    }
    if (ok && warp_wait_bar(&o_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, abort_flag, a.status, 19)) {
      tc_fence_after();
      const float inv = 1.f / l;
      const int qrow = qt * kTcBQ + row;
      f16* orow = a.o + (static_cast<int64_t>(b) * a.n_q + qrow) * a.ldo + h * DH;
      uint32_t o16[16];
#pragma unroll
      for (int c = 0; c < DH / 16; ++c) {
        tmem_ld16(tmem + lane_base + L::kTmemO + 16 * c, o16);
        tmem_ld_wait16(o16);
        float f[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(o16[i]) * inv;
        if (qrow < a.n_q) {
          reinterpret_cast<uint4*>(orow + 16 * c)[0] = pack_f16x8(f);
          reinterpret_cast<uint4*>(orow + 16 * c)[1] = pack_f16x8(f + 8);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
}

// ----------------------------------------------------------------------------
// attn_pp_kernel: two query tiles per CTA, ping-pong between two softmax warpgroups.
//
// One CTA = 256 queries (tiles 0 and 1) of one (sample, head); K/V tiles of 128 keys, shared
// by both query tiles, through a 2-stage TMA ring.  TMEM holds S_0, S_1 (128 fp32 columns
// each) and O_0, O_1 (d_h columns each).  Warps 2-5 run the softmax of tile 0, warps 6-9 of
// tile 1: each reads its S from TMEM (a max pass, then an exp pass), writes P as fp16 pairs
// over the first 64 columns of the same S, and the MMA warp computes O_t += P_t V from
// Tensor Memory (A operand in TMEM), so P needs no shared memory.  The MMA warp issues, per
// key tile j: PV_0(j), S_0(j+1), PV_1(j), S_1(j+1): while one warpgroup runs its softmax,
// the tensor cores work on the other tile.  tcgen05.mma operations of one thread run in
// issue order, so S_t(j+1) overwrites P_t(j) only after PV_t(j) has read it.
// ----------------------------------------------------------------------------
constexpr int kPpThreads = 320;
constexpr int kPpBQ = 256;

// d_h 64 / 128: every 128-row operand tile is d_h / 64 atoms of 64 columns (128-byte swizzle).
// d_h 72: the input heads are padded to 80 columns (columns 72..79 of Q zero), and a tile is
// one 64-column atom plus one 16-column atom (32-byte swizzle); Q K^T runs K = 80 (five
// K = 16 steps), P V runs as an N = 64 and an N = 16 instruction, O keeps 80 TMEM columns of
// which the first 72 are stored.
constexpr int kAtom32 = 128 * 16 * 2;  // 128 rows x 16 fp16: one 32-byte-swizzle column block

template <int DH>
struct PpLayout {
  static constexpr bool kPad = DH == 72;
  static constexpr int kA64 = DH / 64;                // 64-column atoms per tile
  static constexpr int kA16 = kPad ? 1 : 0;           // 16-column atoms per tile
  static constexpr int kDP = 64 * kA64 + 16 * kA16;   // head width the MMAs see
  static constexpr int kTile = kA64 * kAtom + kA16 * kAtom32;
  static constexpr int kQ = 0;                        // Q tile t at kQ + t kTile
  static constexpr int kKV = 2 * kTile;               // stage s: the K tile, then the V tile
  static constexpr int kStage = 2 * kTile;
  static constexpr int kBar = kKV + 2 * kStage;
  static constexpr int kBytes = kBar + 256 + 1024;
  static constexpr uint32_t kTmemS = 0;               // S_t at columns 128 t
  static constexpr uint32_t kTmemO = 256;             // O_t at columns 256 + kDP t
  static_assert(kBytes <= 232448, "shared memory");
  static_assert(kTmemO + 2 * kDP <= 512, "tensor memory");
};

template <int DH>
__global__ void __launch_bounds__(kPpThreads, 1) attn_pp_kernel(const __grid_constant__ AttnTcArgs a) {
  using L = PpLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + L::kBar);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;
  uint64_t* kv_empty = bars + 3;
  uint64_t* s_full = bars + 5;   // per query tile
  uint64_t* p_full = bars + 7;   // per query tile, 4 warps arrive
  uint64_t* o_done = bars + 9;   // per query tile
  uint64_t* drain = bars + 11;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 12);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qt = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.n_heads, h = bh % a.n_heads;
  const int nt = (a.n_kv + kTcBK - 1) / kTcBK;
  // the second query tile of the last pair may hold no query (n_q % 256 in (0, 128], e.g. 258
  // tokens): that CTA then runs tile 0 alone (CTA-uniform)
  const bool two = (2 * qt + 1) * kTcBQ < a.n_q;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], 4);
      mbar_init(&o_done[i], 1);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&a.tmap_q);
    tma_prefetch_desc(&a.tmap_k);
    tma_prefetch_desc(&a.tmap_v);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait_and_trigger();  // the prologue above touched only shared memory and TMEM
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      const int col0 = h * a.head_stride;
      // one 128-row operand tile: its 64-column atoms, then (d_h 72) its 16-column atom
      auto load_tile = [&](uint8_t* dst, const CUtensorMap* m64, const CUtensorMap* m16, uint64_t* bar,
                           int row) {
        for (int at = 0; at < L::kA64; ++at) tma_load_2d(dst + at * kAtom, m64, bar, col0 + at * 64, row);
        if (L::kPad) tma_load_2d(dst + L::kA64 * kAtom, m16, bar, col0 + 64, row);
      };
      mbar_arrive_expect_tx(q_full, (two ? 2 : 1) * L::kTile);
      for (int t = 0; t < (two ? 2 : 1); ++t)
        load_tile(sm + L::kQ + t * L::kTile, &a.tmap_q, &a.tmap_q16, q_full, b * a.n_q + (2 * qt + t) * kTcBQ);
      int j = 0;
      for (; j < nt; ++j) {
        const int s = j & 1;
        if (!mbar_wait(&kv_empty[s], ((j >> 1) & 1) ^ 1u, abort_flag, a.status, 21)) break;
        uint8_t* st = sm + L::kKV + s * L::kStage;
        mbar_arrive_expect_tx(&kv_full[s], 2 * L::kTile);
        const int row = b * a.n_kv + j * kTcBK;
        load_tile(st, &a.tmap_k, &a.tmap_k16, &kv_full[s], row);
        load_tile(st + L::kTile, &a.tmap_v, &a.tmap_v16, &kv_full[s], row);
      }
      if (*abort_flag) {
        drain_bar(q_full, 0);
        for (int i = (j > 2 ? j - 2 : 0); i < j; ++i) drain_bar(&kv_full[i & 1], (i >> 1) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc_qk = umma_idesc_f16(kTcBQ, kTcBK);
      const uint32_t idesc_pv = umma_idesc_f16_bmn(kTcBQ, 64 * L::kA64);
      const uint32_t idesc_pv16 = umma_idesc_f16_bmn(kTcBQ, 16);
      bool ok = mbar_wait(q_full, 0, abort_flag, a.status, 22);
      auto issue_qk = [&](int t, int j) {
        const int s = j & 1;
        const uint32_t qa = smem_u32(sm + L::kQ + t * L::kTile);
        const uint32_t ka = smem_u32(sm + L::kKV + s * L::kStage);
#pragma unroll
        for (int ks = 0; ks < 4 * L::kA64; ++ks) {
          const uint32_t off = (ks >> 2) * kAtom + (ks & 3) * 32;
          umma_f16(tmem + L::kTmemS + t * kTcBK, smem_desc_sw128(qa + off), smem_desc_sw128(ka + off),
                   idesc_qk, ks > 0 ? 1u : 0u);
        }
        if (L::kPad) {  // head columns 64..79 (Q's 72..79 are zero)
          const uint32_t off = L::kA64 * kAtom;
          umma_f16(tmem + L::kTmemS + t * kTcBK, smem_desc_sw32(qa + off), smem_desc_sw32(ka + off),
                   idesc_qk, 1u);
        }
        umma_commit(&s_full[t]);
      };
      auto issue_pv = [&](int t, int j) {
        const int s = j & 1;
        const uint32_t va = smem_u32(sm + L::kKV + s * L::kStage + L::kTile);
#pragma unroll
        for (int ks = 0; ks < kTcBK / 16; ++ks) {
          const uint64_t bd = smem_desc_sw128_mn(va + ks * 2048, kAtom, 1024);
          const uint32_t pa = tmem + L::kTmemS + t * kTcBK + 8 * ks;
          umma_f16_ts(tmem + L::kTmemO + t * L::kDP, pa, bd, idesc_pv, (j > 0 || ks > 0) ? 1u : 0u);
          if (L::kPad) {  // O columns 64..79 from the 16-column V atom (8-key-row groups 256 B apart)
            const uint64_t bd16 = smem_desc_sw32_mn(va + L::kA64 * kAtom + ks * 512, kAtom32, 256);
            umma_f16_ts(tmem + L::kTmemO + t * L::kDP + 64 * L::kA64, pa, bd16, idesc_pv16,
                        (j > 0 || ks > 0) ? 1u : 0u);
          }
        }
        umma_commit(&o_done[t]);
      };
      if (ok && (ok = mbar_wait(&kv_full[0], 0, abort_flag, a.status, 23))) {
        tc_fence_after();
        issue_qk(0, 0);
        if (two) issue_qk(1, 0);
      }
      for (int j = 0; j < nt && ok; ++j) {
        const uint32_t ph = j & 1;
        if (!(ok = mbar_wait(&p_full[0], ph, abort_flag, a.status, 24))) break;
        tc_fence_after();
        issue_pv(0, j);
        if (j + 1 < nt) {
          if (!(ok = mbar_wait(&kv_full[(j + 1) & 1], ((j + 1) >> 1) & 1, abort_flag, a.status, 25))) break;
          tc_fence_after();
          issue_qk(0, j + 1);
        }
        if (two) {
          if (!(ok = mbar_wait(&p_full[1], ph, abort_flag, a.status, 26))) break;
          tc_fence_after();
          issue_pv(1, j);
        }
        umma_commit(&kv_empty[j & 1]);
        if (two && j + 1 < nt) issue_qk(1, j + 1);
      }
      umma_commit(drain);
      drain_bar(drain, 0);
    }
  } else {
    const int t = (warp - 2) >> 2;   // query tile of this warpgroup
    const int q = warp & 3;          // TMEM lane quarter
    const int row = q * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
    const uint32_t s_col = tmem + lane_base + L::kTmemS + t * kTcBK;
    const uint32_t o_col = tmem + lane_base + L::kTmemO + t * L::kDP;
    float m2 = -INFINITY, l = 0.f;
    bool ok = t == 0 || two;  // the warpgroup of an empty second tile has nothing to do
    uint32_t r[kTcBK];
    for (int j = 0; j < nt && ok; ++j) {
      if (!(ok = warp_wait_bar(&s_full[t], j & 1, abort_flag, a.status, 27))) break;
      tc_fence_after();
      const int kb = j * kTcBK;
      const int nvalid = min(a.n_kv - kb, kTcBK);  // keys of this tile (the rest are masked)
      // the whole S row in registers, one TMEM round trip
#pragma unroll
      for (int c = 0; c < kTcBK; c += 16) tmem_ld16(s_col + c, r + c);
#pragma unroll
      for (int c = 0; c < kTcBK; c += 16) tmem_ld_wait16(r + c);
      if (nvalid < kTcBK) {  // masked keys score -inf (P = 0)
#pragma unroll
        for (int c = 0; c < kTcBK; ++c)
          if (c >= nvalid) r[c] = __float_as_uint(-INFINITY);
      }
      // the row maximum of the raw scores (scale > 0 commutes with max), then log2 units
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = __uint_as_float(r[i]);
#pragma unroll
      for (int c = 8; c < kTcBK; ++c) mx[c & 7] = fmaxf(mx[c & 7], __uint_as_float(r[c]));
      const float mt = a.scale_log2 * fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                            fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      if (j == 0) {
        m2 = mt;
      } else if (__any_sync(0xffffffffu, mt > m2 + kRescaleLog2)) {
        // warp-uniform (the TMEM accesses are .sync.aligned); O_t must hold PV_t(j-1)
        if (!(ok = warp_wait_bar(&o_done[t], (j - 1) & 1, abort_flag, a.status, 28))) break;
        tc_fence_after();
        const float mnew = fmaxf(m2, mt);
        const float corr = exp2f(m2 - mnew);
        uint32_t o16[16];
#pragma unroll 1
        for (int c = 0; c < L::kDP; c += 16) {
          tmem_ld16(o_col + c, o16);
          tmem_ld_wait16(o16);
#pragma unroll
          for (int i = 0; i < 16; ++i) o16[i] = __float_as_uint(__uint_as_float(o16[i]) * corr);
          tmem_st16(o_col + c, o16);
        }
        tmem_st_wait();
        l *= corr;
        m2 = mnew;
      }
      // P = 2^(score * scale - m2) packed as fp16 pairs in place (pair k of a 32-score chunk
      // into register k of the chunk, already consumed) and stored over columns [0, 64) of
      // this S: chunk c's 16 packed columns land on scores already read
      const float neg_m2 = -m2;
      float ls[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ls[i] = 0.f;
#pragma unroll
      for (int c = 0; c < kTcBK; c += 32) {
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float p0 = ex2_approx(fmaf(__uint_as_float(r[c + 2 * k]), a.scale_log2, neg_m2));
          const float p1 = ex2_approx(fmaf(__uint_as_float(r[c + 2 * k + 1]), a.scale_log2, neg_m2));
          ls[k & 7] += p0 + p1;
          r[c + k] = pack_f16x2_rn(p0, p1);
        }
        tmem_st16(s_col + c / 2, r + c);
      }
      l += ((ls[0] + ls[1]) + (ls[2] + ls[3])) + ((ls[4] + ls[5]) + (ls[6] + ls[7]));
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[t]);
    }
    if (ok && warp_wait_bar(&o_done[t], (nt - 1) & 1, abort_flag, a.status, 29)) {
      tc_fence_after();
      const float inv = 1.f / l;
      const int qrow = (2 * qt + t) * kTcBQ + row;
      f16* orow = a.o + (static_cast<int64_t>(b) * a.n_q + qrow) * a.ldo + h * DH;
#pragma unroll
      for (int c = 0; c < L::kDP; c += 16) {
        tmem_ld16(o_col + c, r);
        tmem_ld_wait16(r);
        float f[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) f[i] = __uint_as_float(r[i]) * inv;
        if (qrow < a.n_q) {
          reinterpret_cast<uint4*>(orow + c)[0] = pack_f16x8(f);
          if (c + 16 <= DH) reinterpret_cast<uint4*>(orow + c)[1] = pack_f16x8(f + 8);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH>
cudaError_t launch_pp(const AttnPlan& plan, cudaStream_t s) {
  using L = PpLayout<DH>;
  static bool done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(attn_pp_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         L::kBytes);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  const AttnParams& p = plan.p;
  AttnTcArgs a;
  memcpy(&a.tmap_q, &plan.tmap_q, sizeof(CUtensorMap));
  memcpy(&a.tmap_k, &plan.tmap_kv, sizeof(CUtensorMap));
  memcpy(&a.tmap_v, &plan.tmap_v, sizeof(CUtensorMap));
  memcpy(&a.tmap_q16, &plan.tmap_q16, sizeof(CUtensorMap));
  memcpy(&a.tmap_k16, &plan.tmap_k16, sizeof(CUtensorMap));
  memcpy(&a.tmap_v16, &plan.tmap_v16, sizeof(CUtensorMap));
  a.head_stride = p.head_stride > 0 ? p.head_stride : DH;
  a.o = p.o;
  a.ldo = p.ldo;
  a.n_q = p.n_q;
  a.n_kv = p.n_kv;
  a.n_heads = p.n_heads;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
  a.status = device_status_ptr();
  dim3 grid((p.n_q + kPpBQ - 1) / kPpBQ, p.batch * p.n_heads);
  return launch_k(attn_pp_kernel<DH>, grid, dim3(kPpThreads), L::kBytes, s, a);
}

template <int DH>
cudaError_t launch_tc(const AttnPlan& plan, cudaStream_t s) {
  using L = TcLayout<DH>;
  static bool done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         L::kBytes);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  const AttnParams& p = plan.p;
  AttnTcArgs a;
  memcpy(&a.tmap_q, &plan.tmap_q, sizeof(CUtensorMap));
  memcpy(&a.tmap_k, &plan.tmap_kv, sizeof(CUtensorMap));
  memcpy(&a.tmap_v, &plan.tmap_v, sizeof(CUtensorMap));
  a.head_stride = p.head_stride > 0 ? p.head_stride : DH;
  a.o = p.o;
  a.ldo = p.ldo;
  a.n_q = p.n_q;
  a.n_kv = p.n_kv;
  a.n_heads = p.n_heads;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(DH));
  a.status = device_status_ptr();
  dim3 grid((p.n_q + kTcBQ - 1) / kTcBQ, p.batch * p.n_heads);
  return launch_k(attn_tc_kernel<DH>, grid, dim3(kTcThreads), L::kBytes, s, a);
}

template <int DH, int DP>
cudaError_t launch_dh(const AttnParams& p, cudaStream_t s) {
  constexpr int kPitch = DP + 8;
  const int smem = (kBQ + 4 * kBKV) * kPitch * 2;
  static bool done[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64 && !done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<DH, DP>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  dim3 grid((p.n_q + kBQ - 1) / kBQ, p.batch * p.n_heads);
  return launch_k(attn_kernel<DH, DP>, grid, dim3(kWarps * 32), static_cast<size_t>(smem), s, p);
}

}  // namespace

int attn_check(const AttnParams& p, const char** why) {
  if (!p.q || !p.k || !p.v || !p.o || p.batch <= 0 || p.n_q <= 0 || p.n_kv <= 0 ||
      p.n_heads <= 0) {
    *why = "attention: null pointer or empty shape";
    return -1;
  }
  if (!(p.d_head == 64 || p.d_head == 72 || p.d_head == 128)) {
    *why = "attention: d_head must be 64, 72 or 128";
    return -2;
  }
  if ((p.ldq % 8) || (p.ldkv % 8) || (p.ldo % 8) ||
      ((reinterpret_cast<uintptr_t>(p.q) | reinterpret_cast<uintptr_t>(p.k) |
        reinterpret_cast<uintptr_t>(p.v) | reinterpret_cast<uintptr_t>(p.o)) & 15u)) {
    *why = "attention: leading dimensions must be multiples of 8, pointers 16-byte aligned";
    return -2;
  }
  if (p.batch * p.n_heads > 65535) {
    *why = "attention: batch * heads exceeds the grid limit";
    return -2;
  }
  if (p.head_stride != 0 && (p.head_stride < p.d_head || p.head_stride % 8)) {
    *why = "attention: head_stride must be >= d_head and a multiple of 8";
    return -2;
  }
  const int hs = p.head_stride > 0 ? p.head_stride : p.d_head;
  if (p.ldq < (p.n_heads - 1) * hs + p.d_head || p.ldkv < (p.n_heads - 1) * hs + p.d_head) {
    *why = "attention: ldq / ldkv smaller than the heads' columns";
    return -2;
  }
  return 0;
}

int attn_plan(AttnPlan& plan, const char** why) {
  const AttnParams& p = plan.p;
  int rc = attn_check(p, why);
  if (rc) return rc;
  const int hs = p.head_stride > 0 ? p.head_stride : p.d_head;
  // d_h 72 runs on tcgen05 only from a head-padded layout (>= 80 columns per head, Q's
  // columns 72..79 zero), with two query tiles per CTA
  const bool pad72 = p.d_head == 72 && hs >= 80;
  const bool tc_dh = p.d_head == 64 || p.d_head == 128 || (pad72 && p.impl != 2);
  plan.tc = (p.impl == 0 || p.impl == 2 || p.impl == 3) && tc_dh;
  if (!plan.tc) return 0;
  // two query tiles per CTA (ping-pong) unless one tile per CTA is forced: faster on every
  // measured shape, short and ragged ones included (258 tokens: 37.8 against 55.2 us)
  plan.pp = p.impl == 0 || p.impl == 3;
  const int cols = (p.n_heads - 1) * hs + (pad72 ? 80 : p.d_head);
  if (!make_tmap_f16(&plan.tmap_q, p.q, p.batch * p.n_q, cols, p.ldq, kTcBQ) ||
      !make_tmap_f16(&plan.tmap_kv, p.k, p.batch * p.n_kv, cols, p.ldkv, kTcBK) ||
      !make_tmap_f16(&plan.tmap_v, p.v, p.batch * p.n_kv, cols, p.ldkv, kTcBK)) {
    *why = "attention: cuTensorMapEncodeTiled failed";
    return -5;
  }
  if (pad72 && (!make_tmap_f16(&plan.tmap_q16, p.q, p.batch * p.n_q, cols, p.ldq, kTcBQ, 16) ||
                !make_tmap_f16(&plan.tmap_k16, p.k, p.batch * p.n_kv, cols, p.ldkv, kTcBK, 16) ||
                !make_tmap_f16(&plan.tmap_v16, p.v, p.batch * p.n_kv, cols, p.ldkv, kTcBK, 16))) {
    *why = "attention: cuTensorMapEncodeTiled failed";
    return -5;
  }
  return 0;
}

cudaError_t attn_launch(const AttnPlan& plan, cudaStream_t s) {
  const AttnParams& p = plan.p;
  if (plan.tc && plan.pp)
    return p.d_head == 64 ? launch_pp<64>(plan, s) : (p.d_head == 72 ? launch_pp<72>(plan, s) : launch_pp<128>(plan, s));
  if (plan.tc) return p.d_head == 64 ? launch_tc<64>(plan, s) : launch_tc<128>(plan, s);
  switch (p.d_head) {
    case 64: return launch_dh<64, 64>(p, s);
    case 72: return launch_dh<72, 80>(p, s);
    default: return launch_dh<128, 128>(p, s);
  }
}

}  // namespace sgd
