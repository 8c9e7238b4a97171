// Non-causal multi-head attention O = softmax(Q K^T / sqrt(d_h)) V, flash style.
//
// Used inside every active self-attention and cross-attention branch (Algorithm 2:
// an active unit evaluates F_l(h_{l-1,s}; c_s)); frozen units never launch it.
//
// One CTA = 64 query rows of one (sample, head), 4 warps x 16 rows.  K/V tiles of
// 64 keys stream through a double-buffered cp.async ring; S = Q K^T and O += P V run
// on mma.sync m16n8k16 (fp16 in, fp32 accumulate) with an online softmax in
// registers (exp2 with the scale folded in).  Q, K, V, P and O are fp16 (m16n8k16
// f16 x f16 -> f32).  Keys beyond n_kv are masked and their
// shared-memory rows zero-filled; head dims 72 are padded to 80 in shared memory.
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

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int q0 = blockIdx.x * kBQ;
  const int bh = blockIdx.y;
  const int b = bh / p.n_heads, h = bh % p.n_heads;
  const f16* qbase = p.q + (static_cast<int64_t>(b) * p.n_q) * p.ldq + h * DH;
  const f16* kbase = p.k + (static_cast<int64_t>(b) * p.n_kv) * p.ldkv + h * DH;
  const f16* vbase = p.v + (static_cast<int64_t>(b) * p.n_kv) * p.ldkv + h * DH;

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
  attn_kernel<DH, DP><<<grid, kWarps * 32, smem, s>>>(p);
  return cudaGetLastError();
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
  return 0;
}

cudaError_t attn_launch(const AttnParams& p, cudaStream_t s) {
  switch (p.d_head) {
    case 64: return launch_dh<64, 64>(p, s);
    case 72: return launch_dh<72, 80>(p, s);
    default: return launch_dh<128, 128>(p, s);
  }
}

}  // namespace sgd
