// Bandwidth-bound kernels of the scheduled step:
//   frozen_run   — Algorithm 2, frozen branch: h_{l,s} = h_{l-1,s} + Delta_{l, r_l(s)}
//                  for a run of consecutive frozen units in one read-modify-write of h
//                  (16-byte vectors: 8 fp32 of h, 8 fp16 of each cached update).
//   frozen_rows  — the same for models whose pre-norms are folded into the GEMMs, also
//                  writing fp16(h) and the partial row sums the next GEMM normalises with.
//   norm         — pre-norm of an active branch where it cannot be folded (the AdaLN
//                  modulate of DiT-style blocks), fp32 residual in, fp16 GEMM operand out.
//   stem, gemv, head_small, copy_out, pack_f16 — the always-on parts around the
//                  scheduled units (input stage, conditioning, output head, U-ViT skip
//                  operands), Sec. 4.2: conditioning and skip features stay current.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace sgd {

namespace {

constexpr int kNormThreads = 128;
constexpr int kNormMaxVec = 8;  // float4 per thread: d <= 4096

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float s = 0.f;
  const int nw = blockDim.x >> 5;
  for (int i = 0; i < nw; ++i) s += red[i];
  return s;
}

__device__ __forceinline__ void load_bf16x4(const bf16* p, float* f) {
  const uint2 u = *reinterpret_cast<const uint2*>(p);
  const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&u);
  float2 a = __bfloat1622float2(b[0]), c = __bfloat1622float2(b[1]);
  f[0] = a.x; f[1] = a.y; f[2] = c.x; f[3] = c.y;
}

// y = ((x - mean) * rstd) * g + b, then * (1 + scale) + shift (AdaLN), for the 4 columns
// 4 i .. 4 i + 3 of a row; sc / sh point at the row's sample's modulation (or are null).
template <class P>  // NormParams or HeadParams (g, b: bf16 [d] or null)
__device__ __forceinline__ float4 norm_affine4(const P& p, int i, float4 v, float mean, float rstd,
                                               const float* sc, const float* sh) {
  float y[4] = {(v.x - mean) * rstd, (v.y - mean) * rstd, (v.z - mean) * rstd, (v.w - mean) * rstd};
  if (p.g) {
    float g[4];
    load_bf16x4(p.g + 4 * i, g);
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] *= g[k];
  }
  if (p.b) {
    float b[4];
    load_bf16x4(p.b + 4 * i, b);
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] += b[k];
  }
  if (sc) {
    const float4 s4 = *reinterpret_cast<const float4*>(sc + 4 * i);
    const float4 h4 = *reinterpret_cast<const float4*>(sh + 4 * i);
    y[0] = y[0] * (1.f + s4.x) + h4.x;
    y[1] = y[1] * (1.f + s4.y) + h4.y;
    y[2] = y[2] * (1.f + s4.z) + h4.z;
    y[3] = y[3] * (1.f + s4.w) + h4.w;
  }
  return make_float4(y[0], y[1], y[2], y[3]);
}

// The same with the AdaLN modulation read as scalars (any alignment of shift / scale).
__device__ __forceinline__ float4 norm_affine_s(const NormParams& p, int i, float4 v, float mean, float rstd,
                                                const float* sc, const float* sh) {
  float y[4] = {(v.x - mean) * rstd, (v.y - mean) * rstd, (v.z - mean) * rstd, (v.w - mean) * rstd};
  if (p.g) {
    float g[4];
    load_bf16x4(p.g + 4 * i, g);
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] *= g[k];
  }
  if (p.b) {
    float b[4];
    load_bf16x4(p.b + 4 * i, b);
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] += b[k];
  }
  if (sc) {
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] = y[k] * (1.f + sc[4 * i + k]) + sh[4 * i + k];
  }
  return make_float4(y[0], y[1], y[2], y[3]);
}

__device__ __forceinline__ void store_f16x4(f16* p, float4 v) {
  uint2 u;
  u.x = pack_f16x2(v.x, v.y);
  u.y = pack_f16x2(v.z, v.w);
  *reinterpret_cast<uint2*>(p) = u;
}

__global__ void __launch_bounds__(kNormThreads) norm_kernel(const NormParams p) {
  __shared__ float red[kNormThreads / 32];
  pdl_wait_and_trigger();
  const int row = blockIdx.x;
  const int nv = p.d >> 2;
  const float4* hr = reinterpret_cast<const float4*>(p.h + static_cast<int64_t>(row) * p.d);
  float4 v[kNormMaxVec];
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < kNormMaxVec; ++j) {
    const int i = threadIdx.x + j * kNormThreads;
    if (i < nv) {
      v[j] = hr[i];
      sum += (v[j].x + v[j].y) + (v[j].z + v[j].w);
    }
  }
  float mean = 0.f, rstd;
  if (p.kind == SGD_NORM_RMS) {
    float sq = 0.f;
#pragma unroll
    for (int j = 0; j < kNormMaxVec; ++j) {
      const int i = threadIdx.x + j * kNormThreads;
      if (i < nv) sq += (v[j].x * v[j].x + v[j].y * v[j].y) + (v[j].z * v[j].z + v[j].w * v[j].w);
    }
    sq = block_sum(sq, red);
    rstd = rsqrtf(sq / p.d + p.eps);
  } else {
    mean = block_sum(sum, red) / p.d;
    float sq = 0.f;
#pragma unroll
    for (int j = 0; j < kNormMaxVec; ++j) {
      const int i = threadIdx.x + j * kNormThreads;
      if (i < nv) {
        const float a = v[j].x - mean, b = v[j].y - mean, c = v[j].z - mean, d = v[j].w - mean;
        sq += (a * a + b * b) + (c * c + d * d);
      }
    }
    sq = block_sum(sq, red);
    rstd = rsqrtf(sq / p.d + p.eps);
  }
  const float* sh = p.shift ? p.shift + static_cast<int64_t>(row / p.rows_per_batch) * p.ld_mod : nullptr;
  const float* sc = p.scale ? p.scale + static_cast<int64_t>(row / p.rows_per_batch) * p.ld_mod : nullptr;
  f16* orow = p.out + static_cast<int64_t>(row) * p.d;
  // (the fp16 stores cannot alias the fp32 / bf16 parameter loads, so the compiler issues
  // those loads ahead of the stores; transforming every vector before the first store
  // measured slower)
#pragma unroll
  for (int j = 0; j < kNormMaxVec; ++j) {
    const int i = threadIdx.x + j * kNormThreads;
    if (i < nv) store_f16x4(orow + 4 * i, norm_affine_s(p, i, v[j], mean, rstd, sc, sh));
  }
}

// Same normalisation with one warp per row (d <= 2048: at most 16 float4 per lane), one
// row per warp of the block: no block-wide reductions, and for the 1-2 k-wide rows of the mid-size
// models a 128-thread block per row would leave each thread two vectors of work.
constexpr int kNormWarpMaxVec = 16;
__global__ void __launch_bounds__(256) norm_warp_kernel(const NormParams p) {
  pdl_wait_and_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * (blockDim.x >> 5) + warp;
  if (row >= p.rows) return;
  const int nv = p.d >> 2;
  const float4* hr = reinterpret_cast<const float4*>(p.h + static_cast<int64_t>(row) * p.d);
  float4 v[kNormWarpMaxVec];
  float sum = 0.f, sq = 0.f;
#pragma unroll
  for (int j = 0; j < kNormWarpMaxVec; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) {
      v[j] = hr[i];
      sum += (v[j].x + v[j].y) + (v[j].z + v[j].w);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  const float mean = p.kind == SGD_NORM_RMS ? 0.f : sum / p.d;
#pragma unroll
  for (int j = 0; j < kNormWarpMaxVec; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) {
      const float a = v[j].x - mean, b = v[j].y - mean, c = v[j].z - mean, d = v[j].w - mean;
      sq += (a * a + b * b) + (c * c + d * d);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  const float rstd = rsqrtf(sq / p.d + p.eps);
  const float* sh = p.shift ? p.shift + static_cast<int64_t>(row / p.rows_per_batch) * p.ld_mod : nullptr;
  const float* sc = p.scale ? p.scale + static_cast<int64_t>(row / p.rows_per_batch) * p.ld_mod : nullptr;
  f16* orow = p.out + static_cast<int64_t>(row) * p.d;
#pragma unroll
  for (int j = 0; j < kNormWarpMaxVec; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) store_f16x4(orow + 4 * i, norm_affine_s(p, i, v[j], mean, rstd, sc, sh));
  }
}

// Lagged drift of one group's input (App. B.1): each of kDriftBlocks blocks strides over
// float4s of h (two per iteration, to keep more loads in flight), accumulating (h - snap)^2
// and h^2 per thread in fp32, reduces them in a fixed tree and writes its pair; snap takes
// the current h for the next step.  The grid size is fixed, so the summation order (and
// the result) is the same on every run.
__device__ __forceinline__ void drift_acc(const float4 x, const float4 y, float& dd, float& hh) {
  const float a = x.x - y.x, b = x.y - y.y, c = x.z - y.z, d = x.w - y.w;
  dd += (a * a + b * b) + (c * c + d * d);
  hh += (x.x * x.x + x.y * x.y) + (x.z * x.z + x.w * x.w);
}

__global__ void __launch_bounds__(256) drift_kernel(const DriftParams p) {
  __shared__ float red[8];
  pdl_wait_and_trigger();
  const int64_t nv = p.n >> 2;
  const float4* h4 = reinterpret_cast<const float4*>(p.h);
  float4* s4 = reinterpret_cast<float4*>(p.snap);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  float dd = 0.f, hh = 0.f;
  int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (; i + stride < nv; i += 2 * stride) {
    const float4 x0 = h4[i], y0 = s4[i], x1 = h4[i + stride], y1 = s4[i + stride];
    drift_acc(x0, y0, dd, hh);
    drift_acc(x1, y1, dd, hh);
    s4[i] = x0;
    s4[i + stride] = x1;
  }
  if (i < nv) {
    const float4 x = h4[i], y = s4[i];
    drift_acc(x, y, dd, hh);
    s4[i] = x;
  }
  dd = block_sum(dd, red);
  hh = block_sum(hh, red);
  if (threadIdx.x == 0) {
    p.partial[2 * blockIdx.x] = dd;
    p.partial[2 * blockIdx.x + 1] = hh;
  }
}

// One warp per group: lane l sums partials l, l + 32, ... in double, then a fixed xor tree
// combines the lanes (the order is the same on every run).
__global__ void drift_reduce_kernel(const float* partials, double* sums) {
  pdl_wait_and_trigger();
  const float* p = partials + static_cast<size_t>(blockIdx.x) * 2 * kDriftBlocks;
  double dd = 0.0, hh = 0.0;
  for (int b = threadIdx.x; b < kDriftBlocks; b += 32) {
    dd += static_cast<double>(p[2 * b]);
    hh += static_cast<double>(p[2 * b + 1]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    dd += __shfl_xor_sync(0xffffffffu, dd, o);
    hh += __shfl_xor_sync(0xffffffffu, hh, o);
  }
  if (threadIdx.x == 0) {
    sums[2 * blockIdx.x] = dd;
    sums[2 * blockIdx.x + 1] = hh;
  }
}

// Failure-path self-test: thread 0 waits, with the kernels' bounded wait, on an mbarrier
// whose phase nothing completes; after the wait limit it records `code` in the device
// status word and returns.  Used to test the timeout path without faulting the GPU.
__global__ void wait_selftest_kernel(int* status, int code) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, status, code);
}

__global__ void __launch_bounds__(256) frozen_kernel(const __grid_constant__ FrozenParams p) {
  pdl_wait_and_trigger();
  const int64_t n8 = p.n >> 3;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n8; i += stride) {
    float4* hp = reinterpret_cast<float4*>(p.h) + 2 * i;
    const float4 a = hp[0], b = hp[1];
    float acc[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    for (int c = 0; c < p.n_caches; ++c) {
      const uint4 u = __ldcs(reinterpret_cast<const uint4*>(p.caches[c]) + i);
      float f[8];
      unpack_f16x8(u, f);
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[k] += f[k];
    }
    hp[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
    hp[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  }
}

// Frozen run for models whose pre-norms are folded into the GEMMs: also the writer of h's
// fp16 copy and row sums.  Warp w of the grid takes chunk (row, ch) of kStatChunk columns;
// each lane handles 8 consecutive columns per 256-column step, adds the cached updates in
// cache order (the same fp32 arithmetic as frozen_kernel), stores h and fp16(h), and the
// warp reduces its sums with a fixed xor tree into stat slot ch.
__global__ void __launch_bounds__(256) frozen_rows_kernel(const __grid_constant__ FrozenParams p) {
  pdl_wait_and_trigger();
  const int nch = (p.d + kStatChunk - 1) / kStatChunk;
  const int64_t wid = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (wid >= static_cast<int64_t>(p.rows) * nch) return;
  const int lane = threadIdx.x & 31;
  const int row = static_cast<int>(wid / nch), ch = static_cast<int>(wid % nch);
  const int c1 = min(p.d, (ch + 1) * kStatChunk);
  float ss = 0.f, s1 = 0.f;
  for (int c = ch * kStatChunk + lane * 8; c < c1; c += 256) {
    const int64_t i = (static_cast<int64_t>(row) * p.d + c) >> 3;
    float4* hp = reinterpret_cast<float4*>(p.h) + 2 * i;
    const float4 a = hp[0], b = hp[1];
    float acc[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    for (int k = 0; k < p.n_caches; ++k) {
      const uint4 u = __ldcs(reinterpret_cast<const uint4*>(p.caches[k]) + i);
      float f[8];
      unpack_f16x8(u, f);
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] += f[q];
    }
    if (p.n_caches) {
      hp[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
      hp[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
    }
    reinterpret_cast<uint4*>(p.h16)[i] = pack_f16x8(acc);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      ss = fmaf(acc[q], acc[q], ss);
      s1 += acc[q];
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ss += __shfl_xor_sync(0xffffffffu, ss, o);
    s1 += __shfl_xor_sync(0xffffffffu, s1, o);
  }
  if (lane == 0) {
    p.stat[static_cast<int64_t>(ch) * p.rows + row] = ss;
    p.stat[static_cast<int64_t>(kStatSlots + ch) * p.rows + row] = s1;
  }
}

__global__ void io_set_kernel(IoSlot* slot, const IoSlot v) { *slot = v; }

// sinusoid(t, dim)[c] = cos(t w_i) for c < half, sin(t w_{c-half}) otherwise,
// w_i = 10000^(-i / half), evaluated in double precision.
__device__ __forceinline__ float sinusoid_at(double t, int dim, int c) {
  const int half = dim >> 1;
  const int i = c < half ? c : c - half;
  const double w = exp(-9.210340371976184 * static_cast<double>(i) / half);  // ln(10000)
  return static_cast<float>(c < half ? cos(t * w) : sin(t * w));
}

__global__ void stem_kernel(const StemParams p) {
  pdl_wait_and_trigger();
  const int64_t total = static_cast<int64_t>(p.batch) * p.n_tokens * p.d;
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= total) return;
  const int c = static_cast<int>(idx % p.d);
  const int64_t r = idx / p.d;
  const int n = static_cast<int>(r % p.n_tokens);
  const int b = static_cast<int>(r / p.n_tokens);
  const IoSlot* s = p.slot;
  float v = 0.f;
  switch (p.kind) {
    case SGD_STEM_TIME_ADD:
      v = reinterpret_cast<const float*>(s->state)[idx] + sinusoid_at(s->t, p.d, c);
      break;
    case SGD_STEM_IDENTITY:
      v = reinterpret_cast<const float*>(s->state)[idx];
      break;
    case SGD_STEM_EMBED: {
      const int id = min(max(reinterpret_cast<const int32_t*>(s->state)[r], 0), p.vocab - 1);
      v = __bfloat162float(p.embed[static_cast<int64_t>(id) * p.d + c]);
      break;
    }
    case SGD_STEM_PATCH:
    case SGD_STEM_PATCH_TOKENS: {
      const int np = n - p.n_prefix;
      if (np < 0) {
        const int cls = min(max(s->class_ids[b], 0), p.n_classes - 1);
        v = (n == 0) ? sinusoid_at(s->t, p.d, c)
                     : __bfloat162float(p.class_emb[static_cast<int64_t>(cls) * p.d + c]);
      } else {
        const float* z = reinterpret_cast<const float*>(s->state) +
                         (static_cast<int64_t>(b) * (p.n_tokens - p.n_prefix) + np) * p.d_in;
        const bf16* w = p.w_stem + static_cast<int64_t>(c) * p.d_in;
        float acc = 0.f;
        for (int k = 0; k < p.d_in; ++k) acc = fmaf(z[k], __bfloat162float(w[k]), acc);
        v = acc;
      }
      v += __bfloat162float(p.pos[static_cast<int64_t>(n) * p.d + c]);
      break;
    }
    default:
      break;
  }
  p.h[idx] = v;
}

// The patch stems with one thread per (token row, 4 channels): the row's d_in patch values
// and the 4 channels' weight rows are read as 16-byte vectors (d_in % 8 == 0, d % 4 == 0),
// each channel's dot product is summed in k order exactly as in stem_kernel, and the 4
// results go out as one float4.
__global__ void stem_patch_kernel(const StemParams p) {
  pdl_wait_and_trigger();
  const int d4 = p.d >> 2;
  const int64_t total = static_cast<int64_t>(p.batch) * p.n_tokens * d4;
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= total) return;
  const int c0 = static_cast<int>(idx % d4) * 4;
  const int64_t r = idx / d4;
  const int n = static_cast<int>(r % p.n_tokens);
  const int b = static_cast<int>(r / p.n_tokens);
  const IoSlot* s = p.slot;
  float v[4];
  const int np = n - p.n_prefix;
  if (np < 0) {
    const int cls = min(max(s->class_ids[b], 0), p.n_classes - 1);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      v[q] = (n == 0) ? sinusoid_at(s->t, p.d, c0 + q)
                      : __bfloat162float(p.class_emb[static_cast<int64_t>(cls) * p.d + c0 + q]);
  } else {
    const float4* z = reinterpret_cast<const float4*>(
        reinterpret_cast<const float*>(s->state) + (static_cast<int64_t>(b) * (p.n_tokens - p.n_prefix) + np) * p.d_in);
    const uint4* w = reinterpret_cast<const uint4*>(p.w_stem + static_cast<int64_t>(c0) * p.d_in);
    const int w_ld = p.d_in >> 3;  // uint4 per weight row
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = 0.f;
    for (int k8 = 0; k8 < w_ld; ++k8) {
      const float4 za = __ldg(z + 2 * k8), zb = __ldg(z + 2 * k8 + 1);
      const float zf[8] = {za.x, za.y, za.z, za.w, zb.x, zb.y, zb.z, zb.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float wf[8];
        unpack_bf16x8(__ldg(w + q * w_ld + k8), wf);
#pragma unroll
        for (int e = 0; e < 8; ++e) v[q] = fmaf(zf[e], wf[e], v[q]);
      }
    }
  }
  const uint2 pu = __ldg(reinterpret_cast<const uint2*>(p.pos + static_cast<int64_t>(n) * p.d + c0));
  const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&pu);
  const float2 p01 = __bfloat1622float2(pb[0]), p23 = __bfloat1622float2(pb[1]);
  reinterpret_cast<float4*>(p.h)[idx] = make_float4(v[0] + p01.x, v[1] + p01.y, v[2] + p23.x, v[3] + p23.y);
}

// out[r, j] = sum_k act(x[r, k]) W[j, k] for R <= RMAX rows (conditioning and AdaLN
// modulation: a few rows against a large weight, bound by reading W once).  The block stages
// x once in shared memory and then works through output items (32 consecutive columns of one
// segment) with a grid of at most two blocks per SM.  Each warp owns 4 columns of an item; a
// lane streams 16-byte chunks (8 k) of the 4 weight rows and reuses each x chunk across them.
// x is staged as two planes (k % 8 < 4, k % 8 >= 4) so that the lanes' 16-byte x loads are
// consecutive (no bank conflicts).  With 8 rows the warp's 4 x 8 partial sums are reduced by
// a transpose reduction (31 shuffles, lane l ends with value l) instead of 32 butterflies.
constexpr int kGemvCols = 4;

// v[0..31] of every lane -> lane l returns the warp's sum of value l
__device__ __forceinline__ float transpose_reduce32(float* v, int lane) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float a = v[i], b = v[i + o];
      const float send = upper ? a : b;
      v[i] = (upper ? b : a) + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  return v[0];
}

__device__ __forceinline__ void gemv_store(const GemvParams& p, float* out, int r, int j, float v) {
  if (p.add_class) {
    const int cls = min(max(p.slot->class_ids[r], 0), p.n_classes - 1);
    v += __bfloat162float(p.add_class[static_cast<int64_t>(cls) * p.N + j]);
  }
  if (p.add_vec) v += p.add_vec[j];
  out[static_cast<int64_t>(r) * p.ldo + j] = v;
  if (p.out_silu) p.out_silu[static_cast<int64_t>(r) * p.ldo + j] = silu_f(v);
}

template <int RMAX>
__global__ void __launch_bounds__(256) gemv_kernel(const GemvParams p) {
  extern __shared__ float xs[];  // [xrows][2 planes][K / 2]
  pdl_wait_and_trigger();
  const int xrows = p.x_sinusoid ? 1 : (p.ldx == 0 ? 1 : p.rows);
  const int K = p.K, half = K >> 1;
  // x[r][k] lives at r * K + (k & 4 ? half : 0) + (k >> 3) * 4 + (k & 3)
  if (p.x_sinusoid) {
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
      float x = sinusoid_at(p.slot->t, K, k);
      if (p.in_silu) x = silu_f(x);
      xs[((k & 4) ? half : 0) + (k >> 3) * 4 + (k & 3)] = x;
    }
  } else {
    // float4 loads (K % 8 == 0, rows 16-byte aligned) in batches of 8 per thread, every load
    // of a batch issued before its first shared-memory store: x is a generic pointer that
    // the compiler cannot tell apart from xs, so a store in between would make each load
    // wait for the previous element's round trip
    const int k4 = K >> 2, n4 = xrows * k4;
    constexpr int kBatch = 8;
    for (int i0 = threadIdx.x; i0 < n4; i0 += kBatch * blockDim.x) {
      float4 v[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * blockDim.x;
        if (i < n4) {
          const int r = i / k4, k = (i - r * k4) << 2;
          v[j] = __ldg(reinterpret_cast<const float4*>(p.x + static_cast<int64_t>(r) * p.ldx + k));
        }
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * blockDim.x;
        if (i < n4) {
          const int r = i / k4, k = (i - r * k4) << 2;
          float4 x = v[j];
          if (p.in_silu) {
            x.x = silu_f(x.x);
            x.y = silu_f(x.y);
            x.z = silu_f(x.z);
            x.w = silu_f(x.w);
          }
          *reinterpret_cast<float4*>(xs + r * K + ((k & 4) ? half : 0) + (k >> 3) * 4) = x;
        }
      }
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int kItemCols = 8 * kGemvCols;  // 8 warps
  const int per_seg = (p.N + kItemCols - 1) / kItemCols;
  const int n_items = per_seg * (p.n_seg > 0 ? p.n_seg : 1);
  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    const int seg = item / per_seg;
    const int j0 = (item - seg * per_seg) * kItemCols + warp * kGemvCols;
    if (j0 >= p.N) continue;  // warp-uniform; no block-wide barrier follows
    const bf16* W = p.n_seg ? p.w_seg[seg] : p.W;
    float* out = p.n_seg ? p.out_seg[seg] : p.out;
    float acc[kGemvCols * RMAX];
#pragma unroll
    for (int i = 0; i < kGemvCols * RMAX; ++i) acc[i] = 0.f;
    // unrolled so that a warp's weight loads for several K steps are in flight together
#pragma unroll 4
    for (int k = lane * 8; k < K; k += 256) {
      float w[kGemvCols][8];
#pragma unroll
      for (int c = 0; c < kGemvCols; ++c) {
        if (j0 + c < p.N)
          unpack_bf16x8(__ldg(reinterpret_cast<const uint4*>(W + static_cast<int64_t>(j0 + c) * K + k)), w[c]);
        else
#pragma unroll
          for (int q = 0; q < 8; ++q) w[c][q] = 0.f;
      }
      const int xo = (k >> 3) * 4;
#pragma unroll
      for (int r = 0; r < RMAX; ++r) {
        if (r < xrows) {
          const float4 xa = *reinterpret_cast<const float4*>(xs + r * K + xo);
          const float4 xb = *reinterpret_cast<const float4*>(xs + r * K + half + xo);
          const float xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
          for (int c = 0; c < kGemvCols; ++c)
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[c * RMAX + r] = fmaf(w[c][q], xv[q], acc[c * RMAX + r]);
        }
      }
    }
    if constexpr (kGemvCols * RMAX == 32) {
      // lane l: column j0 + l / RMAX, row l % RMAX
      const float v = transpose_reduce32(acc, lane);
      const int c = lane / RMAX, r = lane % RMAX;
      if (r < p.rows && j0 + c < p.N) gemv_store(p, out, r, j0 + c, v);
    } else {
#pragma unroll
      for (int i = 0; i < kGemvCols * RMAX; ++i) {
        if (i % RMAX < xrows) {
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) acc[i] += __shfl_xor_sync(0xffffffffu, acc[i], o);
        }
      }
      if (lane < kGemvCols && j0 + lane < p.N) {
        const int j = j0 + lane;
        // lane c stores column j0 + c; select chains keep acc in registers
        float vals[RMAX];
#pragma unroll
        for (int rr = 0; rr < RMAX; ++rr) {
          float v = acc[rr];
#pragma unroll
          for (int c = 1; c < kGemvCols; ++c) v = (lane == c) ? acc[c * RMAX + rr] : v;
          vals[rr] = v;
        }
        for (int r = 0; r < p.rows; ++r) {
          float v = vals[0];
#pragma unroll
          for (int rr = 1; rr < RMAX; ++rr) v = (xrows > 1 && rr == r) ? vals[rr] : v;
          gemv_store(p, out, r, j, v);
        }
      }
    }
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One warp per row: the fp32 row is read once into registers (lane l holds columns 4 (l + 32 j)
// .. + 3), its mean and rstd are reduced across the warp, the row is normalised (and AdaLN
// modulated) in place, and then every output channel's dot product with it is formed from
// the channel's bf16 weight row (read through the read-only cache: out_channels x K x 2
// bytes, shared by all rows) and reduced across the warp; lane c keeps channel c (and
// c + 32), and the row's outputs are stored together at the end.
template <int MAXV>  // float4 per lane: K <= 128 MAXV
__global__ void __launch_bounds__(256) head_small_kernel(const HeadParams p) {
  pdl_wait_and_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + warp;
  const int64_t rows = static_cast<int64_t>(p.batch) * p.n_tokens;
  if (r >= rows) return;
  const int n = static_cast<int>(r % p.n_tokens), b = static_cast<int>(r / p.n_tokens);
  if (n < p.n_prefix) return;
  float* out = reinterpret_cast<float*>(p.slot->out) +
               (static_cast<int64_t>(b) * (p.n_tokens - p.n_prefix) + (n - p.n_prefix)) *
                   p.out_channels;
  const float4* x = reinterpret_cast<const float4*>(p.h + r * p.ldx);
  const int nv = p.K >> 2;
  float4 v[MAXV];
  float s1 = 0.f;
#pragma unroll
  for (int j = 0; j < MAXV; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) {
      v[j] = __ldg(x + i);
      s1 += (v[j].x + v[j].y) + (v[j].z + v[j].w);
    }
  }
  const float mean = p.norm_kind != SGD_NORM_RMS ? warp_sum(s1) / p.K : 0.f;
  float sq = 0.f;
#pragma unroll
  for (int j = 0; j < MAXV; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) {
      const float a0 = v[j].x - mean, a1 = v[j].y - mean, a2 = v[j].z - mean, a3 = v[j].w - mean;
      sq += (a0 * a0 + a1 * a1) + (a2 * a2 + a3 * a3);
    }
  }
  const float rstd = rsqrtf(warp_sum(sq) / p.K + p.eps);
  const float* sh = p.shift ? p.shift + static_cast<int64_t>(b) * p.ld_mod : nullptr;
  const float* sc = p.scale ? p.scale + static_cast<int64_t>(b) * p.ld_mod : nullptr;
#pragma unroll
  for (int j = 0; j < MAXV; ++j) {
    const int i = lane + 32 * j;
    if (i < nv) v[j] = norm_affine4(p, i, v[j], mean, rstd, sc, sh);
  }
  float res0 = 0.f, res1 = 0.f;
  for (int c = 0; c < p.out_channels; ++c) {
    const uint2* w = reinterpret_cast<const uint2*>(p.W + static_cast<int64_t>(c) * p.K);
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < MAXV; ++j) {
      const int i = lane + 32 * j;
      if (i < nv) {
        const uint2 u = __ldg(w + i);
        const __nv_bfloat162* wb = reinterpret_cast<const __nv_bfloat162*>(&u);
        const float2 w01 = __bfloat1622float2(wb[0]), w23 = __bfloat1622float2(wb[1]);
        acc = fmaf(v[j].x, w01.x, acc);
        acc = fmaf(v[j].y, w01.y, acc);
        acc = fmaf(v[j].z, w23.x, acc);
        acc = fmaf(v[j].w, w23.y, acc);
      }
    }
    acc = warp_sum(acc);
    if (c < 32)
      res0 = lane == c ? acc : res0;
    else
      res1 = lane == c - 32 ? acc : res1;
  }
  if (lane < p.out_channels) out[lane] = res0;
  if (lane + 32 < p.out_channels) out[lane + 32] = res1;
}

__global__ void copy_out_kernel(const IoSlot* slot, const float* h, int64_t n4) {
  pdl_wait_and_trigger();
  float4* o = reinterpret_cast<float4*>(slot->out);
  const float4* s = reinterpret_cast<const float4*>(h);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride)
    o[i] = s[i];
}

__global__ void pack_f16_kernel(f16* dst, int ld_dst, int col0, const float* h, int rows, int d) {
  pdl_wait_and_trigger();
  const int64_t n4 = static_cast<int64_t>(rows) * d / 4;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const int64_t e = i * 4;
    const int64_t r = e / d;
    const int c = static_cast<int>(e % d);
    const float4 v = reinterpret_cast<const float4*>(h)[i];
    uint2 u;
    u.x = pack_f16x2(v.x, v.y);
    u.y = pack_f16x2(v.z, v.w);
    *reinterpret_cast<uint2*>(dst + r * ld_dst + col0 + c) = u;
  }
}

// max |w| over a bf16 tensor: per-block maxima combined with an integer atomicMax on
// the float bit pattern (valid for non-negative floats); *out must start at 0.
__global__ void absmax_bf16_kernel(const bf16* w, int64_t n, float* out) {
  __shared__ float red[8];
  float m = 0.f;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    m = fmaxf(m, fabsf(__bfloat162float(w[i])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < (blockDim.x >> 5); ++i) m = fmaxf(m, red[i]);
    atomicMax(reinterpret_cast<int*>(out), __float_as_int(m));
  }
}

// dst = fp16(w * 2^shift): exact for every bf16 value whose scaled magnitude lies in
// the normal fp16 range (bf16 keeps 8 significant bits, fp16 11).
__global__ void convert_bf16_f16_kernel(const bf16* w, f16* dst, int64_t n, float scale) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    dst[i] = __float2half_rn(sat_f16(__bfloat162float(w[i]) * scale));
}

// max |W[j, k] g[k]| (non-negative floats compared as integers, as absmax_bf16_kernel).
__global__ void absmax_scaled_kernel(const bf16* w, const bf16* g, int64_t n, int K, float* out) {
  __shared__ float red[8];
  float m = 0.f;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    m = fmaxf(m, fabsf(__bfloat162float(w[i]) * __bfloat162float(g[i % K])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < (blockDim.x >> 5); ++i) m = fmaxf(m, red[i]);
    atomicMax(reinterpret_cast<int*>(out), __float_as_int(m));
  }
}

// dst = fp16(W[j, k] g[k] 2^shift): the product of two bf16 values is exact in fp32, and
// is rounded once to fp16.
__global__ void convert_scaled_kernel(const bf16* w, const bf16* g, f16* dst, int64_t n, int K,
                                      float scale) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    dst[i] = __float2half_rn(sat_f16(__bfloat162float(w[i]) * __bfloat162float(g[i % K]) * scale));
}

// One warp per row j: out[j] = scale sum_k W[j, k] (x[k] or 1), accumulated in double.
template <typename TW>
__global__ void rowdot_kernel(const TW* w, const bf16* x, int64_t rows, int K, float scale, float* out) {
  const int64_t j = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (j >= rows) return;
  double acc = 0.0;
  for (int k = lane; k < K; k += 32) {
    const double wv = static_cast<double>(static_cast<float>(w[j * K + k]));
    acc += x ? wv * static_cast<double>(__bfloat162float(x[k])) : wv;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) out[j] = static_cast<float>(acc * scale);
}

__global__ void sampler_kernel(float* z, const float* eps, float alpha, float beta, int64_t n) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += stride)
    z[i] = alpha * z[i] - beta * eps[i];
}

int grid_for(int64_t work, int threads) {
  const int64_t cap = static_cast<int64_t>(num_sms()) * 8;
  int64_t g = (work + threads - 1) / threads;
  if (g > cap) g = cap;
  return g < 1 ? 1 : static_cast<int>(g);
}

}  // namespace

cudaError_t norm_launch(const NormParams& p, cudaStream_t s) {
  // warp per row up to d = 2048; wider rows (LLaDA's 4096) measured faster with the block
  // per row (4.2 against 2.3 TB/s inside the step)
  if (p.d <= 32 * 4 * kNormWarpMaxVec)
    return launch_k(norm_warp_kernel, dim3((p.rows + 7) / 8), dim3(256), 0, s, p);
  else
    return launch_k(norm_kernel, dim3(p.rows), dim3(kNormThreads), 0, s, p);
}

cudaError_t wait_selftest_launch(int* status, int code, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(status, code);
  return cudaGetLastError();
}

cudaError_t drift_launch(const DriftParams& p, cudaStream_t s) {
  return launch_k(drift_kernel, dim3(kDriftBlocks), dim3(256), 0, s, p);
}

cudaError_t drift_reduce_launch(const float* partials, int n_groups, double* sums, cudaStream_t s) {
  return launch_k(drift_reduce_kernel, dim3(n_groups), dim3(32), 0, s, partials, sums);
}

cudaError_t frozen_launch(const FrozenParams& p, cudaStream_t s) {
  if (p.h16) {
    if (!p.stat || p.d % 8 || p.rows < 1 || frozen_stat_slots(p.d) > kStatSlots) return cudaErrorInvalidValue;
    const int64_t warps = static_cast<int64_t>(p.rows) * frozen_stat_slots(p.d);
    return launch_k(frozen_rows_kernel, dim3(static_cast<unsigned>((warps + 7) / 8)), dim3(256), 0, s, p);
  }
  return launch_k(frozen_kernel, dim3(grid_for(p.n / 8, 256)), dim3(256), 0, s, p);
}

cudaError_t io_set_launch(IoSlot* slot, const IoSlot& v, cudaStream_t s) {
  io_set_kernel<<<1, 1, 0, s>>>(slot, v);
  return cudaGetLastError();
}

cudaError_t stem_launch(const StemParams& p, cudaStream_t s) {
  if ((p.kind == SGD_STEM_PATCH || p.kind == SGD_STEM_PATCH_TOKENS) && p.d % 4 == 0 && p.d_in % 8 == 0 &&
      p.d_in > 0) {
    const int64_t total4 = static_cast<int64_t>(p.batch) * p.n_tokens * (p.d / 4);
    return launch_k(stem_patch_kernel, dim3(static_cast<unsigned>((total4 + 255) / 256)), dim3(256), 0, s, p);
  }
  const int64_t total = static_cast<int64_t>(p.batch) * p.n_tokens * p.d;
  return launch_k(stem_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), dim3(256), 0, s, p);
}

template <int RMAX>
cudaError_t gemv_launch_r(const GemvParams& p, size_t smem, cudaStream_t s) {
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(gemv_kernel<RMAX>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  const int cols_per_block = 8 * kGemvCols;
  const int64_t items = static_cast<int64_t>((p.N + cols_per_block - 1) / cols_per_block) * (p.n_seg > 0 ? p.n_seg : 1);
  const int grid = static_cast<int>(std::min<int64_t>(items, 2 * static_cast<int64_t>(num_sms())));
  return launch_k(gemv_kernel<RMAX>, dim3(grid), dim3(256), smem, s, p);
}

cudaError_t gemv_launch(const GemvParams& p, cudaStream_t s) {
  const int xrows = p.x_sinusoid ? 1 : (p.ldx == 0 ? 1 : p.rows);
  const size_t smem = static_cast<size_t>(xrows) * p.K * sizeof(float);
  if (p.rows > 16 || smem > 200 * 1024 || (p.K % 8) || p.n_seg < 0 || p.n_seg > kGemvMaxSeg ||
      (p.n_seg > 0 && (p.out_silu || p.add_class || p.add_vec)) ||
      (!p.x_sinusoid && ((p.ldx % 4) || (reinterpret_cast<uintptr_t>(p.x) & 15u))))
    return cudaErrorInvalidValue;
  if (xrows == 1) return gemv_launch_r<1>(p, smem, s);
  if (xrows <= 8) return gemv_launch_r<8>(p, smem, s);
  return gemv_launch_r<16>(p, smem, s);
}

cudaError_t head_small_launch(const HeadParams& p, cudaStream_t s) {
  const int64_t rows = static_cast<int64_t>(p.batch) * p.n_tokens;
  const dim3 grid(static_cast<unsigned>((rows + 7) / 8));
  if (p.K % 4 || p.K > 4096 || p.out_channels > 64 || p.out_channels > p.N || p.ldx % 4 ||
      (p.shift && p.ld_mod % 4))
    return cudaErrorInvalidValue;
  if (p.K <= 512) return launch_k(head_small_kernel<4>, grid, dim3(256), 0, s, p);
  if (p.K <= 1024) return launch_k(head_small_kernel<8>, grid, dim3(256), 0, s, p);
  if (p.K <= 1536) return launch_k(head_small_kernel<12>, grid, dim3(256), 0, s, p);
  if (p.K <= 2048) return launch_k(head_small_kernel<16>, grid, dim3(256), 0, s, p);
  return launch_k(head_small_kernel<32>, grid, dim3(256), 0, s, p);
}

cudaError_t copy_out_launch(const IoSlot* slot, const float* h, int64_t n, cudaStream_t s) {
  return launch_k(copy_out_kernel, dim3(grid_for(n / 4, 256)), dim3(256), 0, s, slot, h, n / 4);
}

cudaError_t pack_f16_launch(f16* dst, int ld_dst, int col0, const float* h, int rows, int d,
                            cudaStream_t s) {
  return launch_k(pack_f16_kernel, dim3(grid_for(static_cast<int64_t>(rows) * d / 4, 256)), dim3(256), 0, s,
                  dst, ld_dst, col0, h, rows, d);
}

cudaError_t absmax_bf16_launch(const bf16* w, int64_t n, float* out, cudaStream_t s) {
  absmax_bf16_kernel<<<grid_for(n, 256), 256, 0, s>>>(w, n, out);
  return cudaGetLastError();
}

cudaError_t convert_bf16_f16_launch(const bf16* w, f16* dst, int64_t n, int shift, cudaStream_t s) {
  convert_bf16_f16_kernel<<<grid_for(n, 256), 256, 0, s>>>(w, dst, n, ldexpf(1.0f, shift));
  return cudaGetLastError();
}

cudaError_t absmax_scaled_launch(const bf16* w, const bf16* g, int64_t rows, int K, float* out,
                                 cudaStream_t s) {
  absmax_scaled_kernel<<<grid_for(rows * K, 256), 256, 0, s>>>(w, g, rows * K, K, out);
  return cudaGetLastError();
}

cudaError_t convert_scaled_launch(const bf16* w, const bf16* g, f16* dst, int64_t rows, int K, int shift,
                                  cudaStream_t s) {
  convert_scaled_kernel<<<grid_for(rows * K, 256), 256, 0, s>>>(w, g, dst, rows * K, K, ldexpf(1.0f, shift));
  return cudaGetLastError();
}

cudaError_t rowsum_f16_launch(const f16* w, int64_t rows, int K, float scale, float* out, cudaStream_t s) {
  rowdot_kernel<f16><<<static_cast<unsigned>((rows + 7) / 8), 256, 0, s>>>(w, nullptr, rows, K, scale, out);
  return cudaGetLastError();
}

cudaError_t rowdot_bf16_launch(const bf16* w, const bf16* x, int64_t rows, int K, float* out,
                               cudaStream_t s) {
  rowdot_kernel<bf16><<<static_cast<unsigned>((rows + 7) / 8), 256, 0, s>>>(w, x, rows, K, 1.f, out);
  return cudaGetLastError();
}

cudaError_t sampler_launch(float* z, const float* eps, float alpha, float beta, int64_t n,
                           cudaStream_t s) {
  sampler_kernel<<<grid_for(n, 256), 256, 0, s>>>(z, eps, alpha, beta, n);
  return cudaGetLastError();
}

}  // namespace sgd
