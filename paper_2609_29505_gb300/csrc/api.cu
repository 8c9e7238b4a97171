// C ABI of libsgd (include/sgd.h, include/sgd_kernels.h).
//
// sgd_create       borrows the weights, allocates the residual stream and workspaces.
// sgd_set_schedule compiles per-unit lifetimes (Sec. 4.1, Eq. schedule) into the per-step
//                  active/frozen patterns of Sec. 4.2 and captures one CUDA graph per
//                  pattern (plus one per step at which some unit stores its final
//                  update), so that replay has no host branching per layer.
// sgd_step         writes the per-step I/O slot and replays the step's graph
//                  (Algorithm 2).  Inside a graph: stem, conditioning, then for every
//                  unit in graph order either the active branch (norm -> projections
//                  -> attention/MLP -> projection whose epilogue adds Delta to h and,
//                  on the unit's last active step, stores it) or, for a maximal run of
//                  consecutive frozen units, one frozen-run kernel; then the head.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <functional>
#include <map>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/sgd.h"
#include "kernels.h"

using namespace sgd;

namespace sgd {

namespace {
std::vector<unsigned int* (*)()>& clamp_registry() {
  static std::vector<unsigned int* (*)()> r;
  return r;
}
}  // namespace

int register_f16_clamp_flag(unsigned int* (*accessor)()) {
  clamp_registry().push_back(accessor);
  return 1;
}

const std::vector<unsigned int* (*)()>& f16_clamp_flags() { return clamp_registry(); }

bool& pdl_flag() {
  thread_local bool on = false;
  return on;
}

}  // namespace sgd

namespace {

thread_local std::string g_err;

int fail(int code, const std::string& msg) {
  g_err = msg;
  return code;
}

#define CUDA_TRY(expr)                                                                   \
  do {                                                                                   \
    cudaError_t e_ = (expr);                                                             \
    if (e_ != cudaSuccess)                                                               \
      return fail(SGD_ERR_CUDA, std::string(#expr) + ": " + cudaGetErrorString(e_));     \
  } while (0)

struct Op {
  std::string name;
  int kernel;
  double flops;
  double bytes;
  std::function<cudaError_t(cudaStream_t)> run;
};

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int validate_schedule(int T, int n_units, const int32_t* S, const int32_t* groups,
                      int expected_units) {
  if (T < 1) return fail(SGD_ERR_SCHEDULE, "T must be >= 1");
  if (!S || !groups) return fail(SGD_ERR_ARG, "null lifetimes or groups");
  if (expected_units >= 0 && n_units != expected_units)
    return fail(SGD_ERR_SCHEDULE, "n_units " + std::to_string(n_units) + " != model units " +
                                      std::to_string(expected_units));
  if (n_units < 1) return fail(SGD_ERR_SCHEDULE, "n_units must be >= 1");
  std::map<int32_t, int32_t> life_of_group;
  for (int u = 0; u < n_units; ++u) {
    if (S[u] < 1 || S[u] > T)
      return fail(SGD_ERR_SCHEDULE, "lifetime of unit " + std::to_string(u) + " = " +
                                        std::to_string(S[u]) + " outside [1, T]");
    auto it = life_of_group.find(groups[u]);
    if (it == life_of_group.end())
      life_of_group[groups[u]] = S[u];
    else if (it->second != S[u])
      return fail(SGD_ERR_SCHEDULE, "atomic group " + std::to_string(groups[u]) +
                                        " is split: its members have different lifetimes");
  }
  return SGD_OK;
}

// pattern ids in order of first appearance; writes = units whose lifetime ends at s < T
void compile_patterns(int T, int n_units, const int32_t* S, std::vector<int>& pattern_of_step,
                      std::vector<int>& writes, std::vector<std::vector<uint8_t>>& patterns) {
  pattern_of_step.assign(T, 0);
  writes.assign(T, 0);
  patterns.clear();
  std::map<std::vector<uint8_t>, int> ids;
  for (int s = 1; s <= T; ++s) {
    std::vector<uint8_t> m(n_units);
    for (int u = 0; u < n_units; ++u) {
      m[u] = S[u] >= s ? 1 : 0;
      if (S[u] == s && s < T) writes[s - 1]++;
    }
    auto it = ids.find(m);
    if (it == ids.end()) {
      const int id = static_cast<int>(patterns.size());
      ids[m] = id;
      patterns.push_back(m);
      pattern_of_step[s - 1] = id;
    } else {
      pattern_of_step[s - 1] = it->second;
    }
  }
}

}  // namespace

// A GEMM weight as the tensor cores read it: fp16 copy of the user's bf16 matrix scaled
// by 2^shift (exact conversion), with alpha = 2^-shift applied to the accumulator.
struct PW {
  const f16* w = nullptr;
  float alpha = 1.f;
  // pre-norm folded into this weight (its gain multiplied into the columns): LayerNorm
  // column vectors alpha sum_k W'[j, k] and sum_k b_k W[j, k], padded past the last row
  const float* colsum = nullptr;
  const float* colbias = nullptr;
};

struct BlockPW {
  PW qkv, o, xq, xkv, xo, w1, w2;
};

struct sgd_ctx {
  sgd_model_desc d{};
  std::vector<BlockPW> pw;
  std::vector<PW> pw_skip;
  PW pw_head;
  float* absmax = nullptr;
  f16* ctx16 = nullptr;
  std::vector<sgd_block_weights> blk;
  std::vector<const bf16*> skip_w;
  sgd_weights w{};
  int device = 0;
  int M = 0, U = 0, nbr = 0;
  int attn_impl = 0;  // 1: mma.sync attention everywhere (SGD_FLAG_MMA_SYNC_ATTENTION)
  int head_stride = 0;  // columns per head in qkv: d_head, or 80 for d_head 72 on tcgen05
  bool pdl = false;     // programmatic dependent launch between a step program's kernels
  int gemm_bk = 64;   // default K-block of the tcgen05 GEMM
  int exec_mode = SGD_EXEC_JAGGED_GRAPH;
  float* h_pad = nullptr;  // padded mode: residual that discarded branch updates land in
  // pre-norms folded into the GEMMs (RMSNorm / LayerNorm models): every writer of h also
  // writes h16 = fp16(h) and partial row sums into rstat; prog_slots = slots the current
  // writer fills (tracked while a step program is built)
  bool fold = false;
  f16* h16 = nullptr;
  float* rstat = nullptr;
  float* rstat_final = nullptr;  // row totals finalised by a writer GEMM (slot 0)
  int* stat_cnt = nullptr;       // per 128-row block tickets of that finalisation
  const float* prog_stat = nullptr;  // statistics buffer of the current writer of h
  int prog_slots = 0;
  // stream-K GEMM workspace, shared by every GEMM of this context (they run one after
  // another on one stream); grown when a new plan needs more, the old buffers stay
  // allocated for graphs captured with them
  float* sk_ws = nullptr;
  int* sk_cnt = nullptr;
  size_t sk_ws_floats = 0, sk_need_floats = 0;
  int sk_cnt_n = 0, sk_need_cnt = 0;
  // buffers
  float* h = nullptr;
  f16* xn = nullptr;
  f16* qkv = nullptr;
  f16* attn = nullptr;
  f16* act = nullptr;
  float* t_hidden = nullptr;
  float* cond_c = nullptr;
  float* cond_silu = nullptr;
  float* mod = nullptr;
  float* modf = nullptr;
  float* rope_cos = nullptr;
  float* rope_sin = nullptr;
  IoSlot* slot = nullptr;
  std::vector<f16*> cache;
  std::vector<f16*> ctxkv;
  std::vector<f16*> skipcat;
  std::vector<void*> allocs;
  size_t cache_bytes = 0, ws_bytes = 0, weight_bytes = 0;
  // schedule
  int T = 0;
  std::vector<int32_t> S, groups;
  std::vector<int> pattern_of_step, writes;
  std::vector<std::vector<uint8_t>> patterns;
  std::vector<int> graph_of_step;
  std::vector<std::vector<Op>> programs;
  std::vector<cudaGraph_t> graphs;
  std::vector<cudaGraphExec_t> execs;
  cudaStream_t cap_stream = nullptr;
  int last_step = 0;
  bool scheduled = false;
  // host-buffer step staging
  void* st_in = nullptr;
  void* st_out = nullptr;
  int32_t* st_cls = nullptr;
  void* st_ctx = nullptr;
  // asynchronous host-buffer steps: double-buffered device output, copy stream, events
  void* st_out2[2] = {nullptr, nullptr};
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t ev_done[2] = {nullptr, nullptr};
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};
  cudaEvent_t ev_last = nullptr;  // the last host-mapped step (sgd_host_wait)
  bool ev_last_used = false;
  int async_slot = 0;
  // input-aware (drift) policy, App. B.1
  int policy = SGD_POLICY_STATIC;
  int n_groups = 0;
  std::vector<int> group_of_unit;    // group index (groups numbered by their first unit)
  std::vector<uint8_t> group_start;  // 1 for the first unit of each group
  std::vector<int> m_of_step;        // static active-group count at steps 1..T
  float* snap = nullptr;             // [G][M d] fp32: each group's input at the last step
  float* drift_part = nullptr;       // [G][kDriftBlocks][2]
  double* drift_sums = nullptr;      // [G][2]: sum (h - snap)^2, sum h^2
  double* drift_host = nullptr;      // pinned copy of drift_sums
  size_t drift_alloc_groups = 0;
  cudaEvent_t ev_drift = nullptr;    // recorded after the copy of a step's drift sums
  std::map<std::vector<uint8_t>, int> drift_graph_of;            // library: pattern -> graph
  std::map<std::vector<uint8_t>, std::vector<Op>> drift_eager;   // patterns outside it
  std::vector<std::vector<double>> drift_used;  // [T + 1]: drifts ranked at each step
  std::vector<std::vector<uint8_t>> mask_used;  // [T + 1]: unit mask each step ran
  int64_t graph_steps = 0, eager_steps = 0;

  ~sgd_ctx() {
    if (ev_last_used) cudaEventSynchronize(ev_last);
    if (copy_stream) cudaStreamSynchronize(copy_stream);
    if (ev_drift) cudaEventDestroy(ev_drift);
    if (drift_host) cudaFreeHost(drift_host);
    for (int i = 0; i < 2; ++i) {
      if (ev_done[i]) cudaEventDestroy(ev_done[i]);
      if (ev_copied[i]) cudaEventDestroy(ev_copied[i]);
    }
    if (ev_last) cudaEventDestroy(ev_last);
    if (copy_stream) cudaStreamDestroy(copy_stream);
    for (auto e : execs) cudaGraphExecDestroy(e);
    for (auto g : graphs) cudaGraphDestroy(g);
    if (cap_stream) cudaStreamDestroy(cap_stream);
    for (void* p : allocs) cudaFree(p);
  }

  template <typename T_>
  int alloc(T_** p, size_t count, size_t* acct) {
    void* q = nullptr;
    const size_t bytes = std::max<size_t>(count * sizeof(T_), 16);
    cudaError_t e = cudaMalloc(&q, bytes);
    if (e != cudaSuccess)
      return fail(e == cudaErrorMemoryAllocation ? SGD_ERR_OOM : SGD_ERR_CUDA,
                  std::string("cudaMalloc: ") + cudaGetErrorString(e));
    allocs.push_back(q);
    if (acct) *acct += bytes;
    *p = static_cast<T_*>(q);
    return SGD_OK;
  }

  size_t in_bytes() const {
    if (d.stem == SGD_STEM_EMBED) return static_cast<size_t>(M) * 4;
    return static_cast<size_t>(d.batch) * (d.n_tokens - d.n_prefix) * d.d_in * 4;
  }
  size_t out_bytes() const {
    if (d.head == SGD_HEAD_LOGITS) return static_cast<size_t>(M) * d.d_out * 2;  // fp16 logits
    if (d.head == SGD_HEAD_IDENTITY) return static_cast<size_t>(M) * d.d * 4;
    return static_cast<size_t>(d.batch) * (d.n_tokens - d.n_prefix) * d.out_channels * 4;
  }
};

namespace {

const bf16* B16(const void* p) { return static_cast<const bf16*>(p); }
const f16* H16(const void* p) { return static_cast<const f16*>(p); }

// ---------------------------------------------------------------------------
// op builders
// ---------------------------------------------------------------------------

int make_gemm_op(sgd_ctx* c, std::vector<Op>& ops, const std::string& name, const f16* A,
                 int lda, const PW& B, int ldb, int M, int N, int K, EpiParams epi) {
  epi.alpha = B.alpha;
  if (epi.norm == SGD_FNORM_LN) {
    epi.colsum = B.colsum;
    epi.colbias = B.colbias;
  }
  auto plan = std::make_shared<GemmPlan>();
  plan->A = A;
  plan->lda = lda;
  plan->B = B.w;
  plan->ldb = ldb;
  plan->M = M;
  plan->N = N;
  plan->K = K;
  plan->epi = epi;
  plan->simt = (c->d.flags & SGD_FLAG_SIMT_GEMM) != 0;
  plan->bk = (c->d.flags & SGD_FLAG_GEMM_BK64) ? 64 : c->gemm_bk;
  const char* why = "";
  if (gemm_plan(*plan, &why) != 0) return fail(SGD_ERR_SHAPE, std::string(name) + ": " + why);
  plan->ws_ref = &c->sk_ws;
  plan->cnt_ref = &c->sk_cnt;
  c->sk_need_floats = std::max(c->sk_need_floats, gemm_ws_floats(*plan));
  c->sk_need_cnt = std::max(c->sk_need_cnt, plan->sk_tiles);
  const bool gated = epi.kind == SGD_EPI_GATED;
  const double nb = gated ? 2.0 * N : N;
  double out_b;
  switch (epi.kind) {
    case SGD_EPI_F32: out_b = 4.0 * M * N; break;
    case SGD_EPI_DELTA: out_b = 8.0 * M * N + (epi.cache ? 2.0 * M * N : 0.0); break;
    default: out_b = 2.0 * M * N; break;
  }
  if (epi.h16) {  // writer of h: its fp16 copy and row sums (slots of this plan's column tiles)
    const int num_n = (N + plan->bn - 1) / plan->bn;
    out_b += 2.0 * M * N + 16.0 * M * num_n;
    if (epi.stat_cnt) {  // finalised by the writer: the next GEMM reads one slot
      c->prog_stat = epi.stat_final;
      c->prog_slots = 1;
    } else {
      c->prog_stat = epi.stat_out;
      c->prog_slots = 2 * num_n;
    }
  }
  if (epi.norm != SGD_FNORM_NONE) out_b += 8.0 * M * epi.stat_slots * (epi.norm == SGD_FNORM_LN ? 2 : 1);
  Op op;
  op.name = name;
  op.kernel = plan->simt ? SGD_KERNEL_GEMM_SIMT : SGD_KERNEL_GEMM_TC;
  op.flops = 2.0 * M * nb * K;
  op.bytes = 2.0 * M * K + 2.0 * nb * K + out_b;
  op.run = [plan](cudaStream_t s) { return gemm_launch(*plan, s); };
  ops.push_back(std::move(op));
  return SGD_OK;
}

EpiParams epi_base(int kind) {
  EpiParams e{};
  e.kind = kind;
  e.alpha = 1.f;
  e.rows_per_batch = 1;
  return e;
}

// The GEMM that follows a folded pre-norm: A is h16, the epilogue normalises each row with
// the statistics of the current writer of h.
void set_folded_norm(sgd_ctx* c, EpiParams& e, int norm_kind) {
  e.norm = norm_kind == SGD_NORM_RMS ? SGD_FNORM_RMS : SGD_FNORM_LN;
  e.rstat = c->prog_stat;
  e.stat_slots = c->prog_slots;
  e.stat_ld = c->M;
  e.norm_eps = c->d.eps;
  e.norm_inv_d = 1.0f / static_cast<float>(c->d.d);
}

// A GEMM epilogue that writes h also writes h16 and the row sums.
void set_h_writer(sgd_ctx* c, EpiParams& e) {
  e.h16 = c->h16;
  e.stat_out = c->rstat;
  e.stat_out_ld = c->M;
  e.stat_cnt = c->stat_cnt;
  e.stat_final = c->rstat_final;
}

// h16 and row sums of h as it stands (after the stem): a frozen run of no units.
void make_hstat_op(sgd_ctx* c, std::vector<Op>& ops) {
  FrozenParams p{};
  p.h = c->h;
  p.n = static_cast<int64_t>(c->M) * c->d.d;
  p.rows = c->M;
  p.d = c->d.d;
  p.h16 = c->h16;
  p.stat = c->rstat;
  Op op;
  op.name = "h_stats";
  op.kernel = SGD_KERNEL_FROZEN_RUN;
  op.flops = 2.0 * p.n;
  op.bytes = 6.0 * p.n;
  op.run = [p](cudaStream_t s) { return frozen_launch(p, s); };
  ops.push_back(std::move(op));
  c->prog_stat = c->rstat;
  c->prog_slots = frozen_stat_slots(c->d.d);
}

void make_norm_op(sgd_ctx* c, std::vector<Op>& ops, const std::string& name, int kind,
                  const void* g, const void* b, const float* shift, const float* scale, int ld_mod) {
  NormParams p{};
  p.h = c->h;
  p.out = c->xn;
  p.rows = c->M;
  p.d = c->d.d;
  p.kind = kind;
  p.g = B16(g);
  p.b = B16(b);
  p.shift = shift;
  p.scale = scale;
  p.ld_mod = ld_mod;
  p.rows_per_batch = c->d.n_tokens;
  p.eps = c->d.eps;
  Op op;
  op.name = name;
  op.kernel = SGD_KERNEL_NORM;
  op.flops = 0;
  op.bytes = 6.0 * c->M * c->d.d;
  op.run = [p](cudaStream_t s) { return norm_launch(p, s); };
  ops.push_back(std::move(op));
}

int make_attn_op(sgd_ctx* c, std::vector<Op>& ops, const std::string& name, const AttnParams& p) {
  const char* why = "";
  auto plan = std::make_shared<AttnPlan>();
  plan->p = p;
  if (attn_plan(*plan, &why) != 0) return fail(SGD_ERR_SHAPE, name + ": " + why);
  Op op;
  op.name = name;
  op.kernel = SGD_KERNEL_ATTENTION;
  const double dm = static_cast<double>(p.n_heads) * p.d_head;
  op.flops = 4.0 * p.batch * p.n_heads * static_cast<double>(p.n_q) * p.n_kv * p.d_head;
  op.bytes = 2.0 * p.batch * (2.0 * p.n_q * dm + 2.0 * p.n_kv * dm);
  op.run = [plan](cudaStream_t s) { return attn_launch(*plan, s); };
  ops.push_back(std::move(op));
  return SGD_OK;
}

void make_gemv_op(std::vector<Op>& ops, const std::string& name, const GemvParams& p) {
  Op op;
  op.name = name;
  op.kernel = SGD_KERNEL_SMALL;
  const double seg = p.n_seg > 0 ? p.n_seg : 1;
  op.flops = 2.0 * seg * p.rows * p.N * p.K;
  op.bytes = seg * (2.0 * p.N * p.K + 4.0 * p.rows * p.N) + 4.0 * p.rows * p.K;
  op.run = [p](cudaStream_t s) { return gemv_launch(p, s); };
  ops.push_back(std::move(op));
}

void flush_run(sgd_ctx* c, std::vector<Op>& ops, std::vector<const f16*>& run, int first_unit) {
  size_t i = 0;
  while (i < run.size()) {
    FrozenParams p{};
    p.h = c->h;
    p.n = static_cast<int64_t>(c->M) * c->d.d;
    p.n_caches = 0;
    p.rows = c->M;
    p.d = c->d.d;
    if (c->fold) {
      p.h16 = c->h16;
      p.stat = c->rstat;
      c->prog_stat = c->rstat;
      c->prog_slots = frozen_stat_slots(c->d.d);
    }
    while (i < run.size() && p.n_caches < kMaxRun) p.caches[p.n_caches++] = run[i++];
    Op op;
    op.name = "frozen_run(u" + std::to_string(first_unit) + "+" + std::to_string(p.n_caches) + ")";
    op.kernel = SGD_KERNEL_FROZEN_RUN;
    op.flops = static_cast<double>(p.n) * p.n_caches;
    op.bytes = static_cast<double>(p.n) * (8.0 + 2.0 * p.n_caches + (c->fold ? 2.0 : 0.0));
    op.run = [p](cudaStream_t s) { return frozen_launch(p, s); };
    ops.push_back(std::move(op));
  }
  run.clear();
}

int build_branch(sgd_ctx* c, std::vector<Op>& ops, int b, int kind, bool write_cache, int u,
                 bool discard = false) {
  const sgd_model_desc& d = c->d;
  const sgd_block_weights& W = c->blk[b];
  const BlockPW& P = c->pw[b];
  const int M = c->M, D = d.d, F = d.d_ff;
  const std::string pre = "b" + std::to_string(b) + ".";
  const bool adaln = d.block == SGD_BLOCK_ADALN;
  float* mod = adaln ? c->mod + static_cast<size_t>(b) * d.batch * 6 * D : nullptr;
  f16* cache = write_cache ? c->cache[u] : nullptr;
  EpiParams delta = epi_base(SGD_EPI_DELTA);
  delta.h = discard ? c->h_pad : c->h;
  delta.ldh = D;
  delta.cache = discard ? nullptr : cache;
  delta.ld_cache = D;
  if (c->fold && !discard) set_h_writer(c, delta);
  // the pre-norm's input: h16 with the norm folded into the GEMM, else the norm kernel's output
  const f16* xin = c->fold ? c->h16 : c->xn;
  int rc;
  if (kind == 0) {  // self-attention
    if (!c->fold)
      make_norm_op(c, ops, pre + "attn.norm", d.norm, W.norm1_w, W.norm1_b, adaln ? mod : nullptr,
                   adaln ? mod + D : nullptr, 6 * D);
    EpiParams e = epi_base(d.rope ? SGD_EPI_ROPE : SGD_EPI_F16);
    if (c->fold) set_folded_norm(c, e, d.norm);
    const int HS = c->head_stride, QW = d.n_heads * HS;  // qkv: [M, 3 QW], head h of Q at h HS
    e.out = c->qkv;
    e.ldo = 3 * QW;
    if (HS != d.d_head) {
      e.pad_src = d.d_head;
      e.pad_dst = HS;
    }
    if (d.rope) {
      e.rope_cos = c->rope_cos;
      e.rope_sin = c->rope_sin;
      e.rope_tokens = d.n_tokens;
      e.d_head = d.d_head;
      e.rope_cols = 2 * D;
    }
    if ((rc = make_gemm_op(c, ops, pre + "attn.qkv", xin, D, P.qkv, D, M, 3 * D, D, e)))
      return rc;
    AttnParams ap{c->qkv, 3 * QW, c->qkv + QW, c->qkv + 2 * QW, 3 * QW, c->attn, D,
                  d.batch, d.n_tokens, d.n_tokens, d.n_heads, d.d_head, c->attn_impl, HS};
    if ((rc = make_attn_op(c, ops, pre + "attn.sdpa", ap))) return rc;
    if (adaln) {
      delta.gate = mod + 2 * D;
      delta.ld_gate = 6 * D;
      delta.rows_per_batch = d.n_tokens;
    }
    return make_gemm_op(c, ops, pre + "attn.out", c->attn, D, P.o, D, M, D, D, delta);
  }
  if (kind == 1) {  // cross-attention
    if (!c->fold)
      make_norm_op(c, ops, pre + "xattn.norm", SGD_NORM_LN, W.normx_w, W.normx_b, nullptr, nullptr, 0);
    EpiParams e = epi_base(SGD_EPI_F16);
    if (c->fold) set_folded_norm(c, e, SGD_NORM_LN);
    e.out = c->qkv;
    e.ldo = D;
    if ((rc = make_gemm_op(c, ops, pre + "xattn.q", xin, D, P.xq, D, M, D, D, e))) return rc;
    AttnParams ap{c->qkv, D, c->ctxkv[b], c->ctxkv[b] + D, 2 * D, c->attn, D,
                  d.batch, d.n_tokens, d.ctx_len, d.n_heads, d.d_head, c->attn_impl, 0};
    if ((rc = make_attn_op(c, ops, pre + "xattn.sdpa", ap))) return rc;
    return make_gemm_op(c, ops, pre + "xattn.out", c->attn, D, P.xo, D, M, D, D, delta);
  }
  // MLP
  if (!c->fold)
    make_norm_op(c, ops, pre + "mlp.norm", d.norm, W.norm2_w, W.norm2_b, adaln ? mod + 3 * D : nullptr,
                 adaln ? mod + 4 * D : nullptr, 6 * D);
  const bool gated = d.mlp == SGD_MLP_SWIGLU || d.mlp == SGD_MLP_GEGLU;
  EpiParams e = epi_base(gated ? SGD_EPI_GATED : SGD_EPI_GELU);
  if (c->fold) set_folded_norm(c, e, d.norm);
  e.out = c->act;
  e.ldo = F;
  e.act = (d.mlp == SGD_MLP_GEGLU || d.mlp == SGD_MLP_GELU_ERF) ? 1 : 0;
  if ((rc = make_gemm_op(c, ops, pre + "mlp.up", xin, D, P.w1, D, M, F, D, e))) return rc;
  if (adaln) {
    delta.gate = mod + 5 * D;
    delta.ld_gate = 6 * D;
    delta.rows_per_batch = d.n_tokens;
  }
  return make_gemm_op(c, ops, pre + "mlp.down", c->act, F, P.w2, F, M, D, F, delta);
}

int build_program(sgd_ctx* c, const std::vector<uint8_t>& active, const std::vector<uint8_t>& write,
                  std::vector<Op>& ops) {
  const sgd_model_desc& d = c->d;
  const int M = c->M, D = d.d;
  ops.clear();
  int rc;
  {  // stem
    StemParams p{};
    p.kind = d.stem;
    p.slot = c->slot;
    p.h = c->h;
    p.batch = d.batch;
    p.n_tokens = d.n_tokens;
    p.n_prefix = d.n_prefix;
    p.d = D;
    p.d_in = d.d_in;
    p.w_stem = B16(c->w.w_stem);
    p.pos = B16(c->w.pos_emb);
    p.class_emb = B16(c->w.class_emb);
    p.embed = B16(c->w.embed);
    p.vocab = d.vocab;
    p.n_classes = d.n_classes;
    Op op;
    op.name = "stem";
    op.kernel = SGD_KERNEL_SMALL;
    op.flops = 2.0 * M * D * std::max(d.d_in, 1);
    op.bytes = 4.0 * M * D + static_cast<double>(c->in_bytes()) +
               (d.stem == SGD_STEM_EMBED ? 2.0 * M * D : 0.0);
    op.run = [p](cudaStream_t s) { return stem_launch(p, s); };
    ops.push_back(std::move(op));
    if (c->fold) make_hstat_op(c, ops);
  }
  if (d.block == SGD_BLOCK_ADALN) {  // conditioning: c = W_t2 silu(W_t1 sin(t)) + class_emb[y]
    GemvParams g{};
    g.out = c->t_hidden;
    g.ldo = D;
    g.x_sinusoid = 1;
    g.slot = c->slot;
    g.W = B16(c->w.w_t1);
    g.N = D;
    g.K = d.t_freq;
    g.rows = 1;
    make_gemv_op(ops, "cond.t1", g);
    GemvParams g2{};
    g2.out = c->cond_c;
    g2.ldo = D;
    g2.x = c->t_hidden;
    g2.ldx = 0;
    g2.slot = c->slot;
    g2.in_silu = 1;
    g2.W = B16(c->w.w_t2);
    g2.N = D;
    g2.K = D;
    g2.rows = d.batch;
    g2.add_class = B16(c->w.class_emb);
    g2.n_classes = d.n_classes;
    g2.out_silu = c->cond_silu;
    make_gemv_op(ops, "cond.t2", g2);
    // the modulation (shift, scale, gate: rows 3 D k .. 3 D k + 3 D of W_mod) of every active
    // branch k of every block, in one launch: it depends on c only, and per-block launches of
    // a 16 MB weight each left most of the GPU idle
    GemvParams gm{};
    gm.ldo = 6 * D;
    gm.x = c->cond_silu;
    gm.ldx = D;
    gm.slot = c->slot;
    gm.in_silu = 0;
    gm.N = 3 * D;
    gm.K = D;
    gm.rows = d.batch;
    for (int b = 0; b < d.n_blocks; ++b) {
      for (int k = 0; k < c->nbr; ++k) {
        if (!active[b * c->nbr + k]) continue;  // modulation only for active branches
        gm.w_seg[gm.n_seg] = B16(c->blk[b].w_mod) + static_cast<size_t>(k) * 3 * D * D;
        gm.out_seg[gm.n_seg] = c->mod + static_cast<size_t>(b) * d.batch * 6 * D + static_cast<size_t>(k) * 3 * D;
        if (++gm.n_seg == kGemvMaxSeg) {
          make_gemv_op(ops, "mod", gm);
          gm.n_seg = 0;
        }
      }
    }
    if (gm.n_seg > 0) make_gemv_op(ops, "mod", gm);
  }
  std::vector<const f16*> run;
  int run_first = 0;
  int u = 0;
  for (int b = 0; b < d.n_blocks; ++b) {
    if (d.n_skips && b > d.n_skips) {  // U-ViT deep block: h = W_skip [h; skip]
      flush_run(c, ops, run, run_first);
      const int j = b - d.n_skips - 1;
      f16* cat = c->skipcat[j];
      const float* hh = c->h;
      const int Mr = M;
      Op op;
      op.name = "b" + std::to_string(b) + ".skip_pack";
      op.kernel = SGD_KERNEL_SMALL;
      op.flops = 0;
      op.bytes = 6.0 * M * D;
      op.run = [cat, hh, Mr, D](cudaStream_t s) { return pack_f16_launch(cat, 2 * D, 0, hh, Mr, D, s); };
      ops.push_back(std::move(op));
      EpiParams e = epi_base(SGD_EPI_F32);
      e.out = c->h;
      e.ldo = D;
      if (c->fold) set_h_writer(c, e);
      if ((rc = make_gemm_op(c, ops, "b" + std::to_string(b) + ".skip_linear", cat, 2 * D,
                             c->pw_skip[j], 2 * D, M, D, 2 * D, e)))
        return rc;
    }
    for (int k = 0; k < c->nbr; ++k, ++u) {
      const int kind = d.block == SGD_BLOCK_XATTN ? k : (k == 0 ? 0 : 2);
      if (c->policy == SGD_POLICY_DRIFT && c->group_start[u]) {
        // App. B.1: lagged drift of the group's input (the stream entering its first branch)
        flush_run(c, ops, run, run_first);
        const int g = c->group_of_unit[u];
        DriftParams dp{c->h, c->snap + static_cast<size_t>(g) * M * D, static_cast<int64_t>(M) * D,
                       c->drift_part + static_cast<size_t>(g) * 2 * kDriftBlocks};
        Op op;
        op.name = "g" + std::to_string(g) + ".drift";
        op.kernel = SGD_KERNEL_SMALL;
        op.flops = 4.0 * M * D;
        op.bytes = 12.0 * M * D;
        op.run = [dp](cudaStream_t s) { return drift_launch(dp, s); };
        ops.push_back(std::move(op));
      }
      if (active[u]) {
        flush_run(c, ops, run, run_first);
        if ((rc = build_branch(c, ops, b, kind, write[u] != 0, u))) return rc;
      } else {
        if (c->exec_mode == SGD_EXEC_PADDED_GRAPH) {
          // padded execution: the frozen branch is evaluated anyway and its update discarded
          flush_run(c, ops, run, run_first);
          if ((rc = build_branch(c, ops, b, kind, false, u, true))) return rc;
        }
        if (run.empty()) run_first = u;
        run.push_back(c->cache[u]);
      }
    }
    if (d.n_skips && b < d.n_skips) {  // U-ViT shallow block: push the current h
      flush_run(c, ops, run, run_first);
      f16* cat = c->skipcat[d.n_skips - 1 - b];
      const float* hh = c->h;
      const int Mr = M;
      Op op;
      op.name = "b" + std::to_string(b) + ".skip_push";
      op.kernel = SGD_KERNEL_SMALL;
      op.flops = 0;
      op.bytes = 6.0 * M * D;
      op.run = [cat, hh, Mr, D](cudaStream_t s) { return pack_f16_launch(cat, 2 * D, D, hh, Mr, D, s); };
      ops.push_back(std::move(op));
    }
  }
  flush_run(c, ops, run, run_first);
  if (c->policy == SGD_POLICY_DRIFT) {
    const float* part = c->drift_part;
    double* sums = c->drift_sums;
    const int G = c->n_groups;
    Op op;
    op.name = "drift.reduce";
    op.kernel = SGD_KERNEL_SMALL;
    op.flops = 0;
    op.bytes = 8.0 * G * kDriftBlocks;
    op.run = [part, G, sums](cudaStream_t s) { return drift_reduce_launch(part, G, sums, s); };
    ops.push_back(std::move(op));
  }
  // head
  void* const* out_slot = reinterpret_cast<void* const*>(&c->slot->out);
  if (d.head == SGD_HEAD_IDENTITY) {
    const IoSlot* slot = c->slot;
    const float* hh = c->h;
    const int64_t n = static_cast<int64_t>(M) * D;
    Op op;
    op.name = "head.copy";
    op.kernel = SGD_KERNEL_SMALL;
    op.flops = 0;
    op.bytes = 8.0 * n;
    op.run = [slot, hh, n](cudaStream_t s) { return copy_out_launch(slot, hh, n, s); };
    ops.push_back(std::move(op));
    return SGD_OK;
  }
  const float* shift = nullptr;
  const float* scale = nullptr;
  if (d.head == SGD_HEAD_ADALN_LINEAR) {
    GemvParams g{};
    g.out = c->modf;
    g.ldo = 2 * D;
    g.x = c->cond_silu;
    g.ldx = D;
    g.slot = c->slot;
    g.in_silu = 0;
    g.W = B16(c->w.w_modf);
    g.N = 2 * D;
    g.K = D;
    g.rows = d.batch;
    make_gemv_op(ops, "head.mod", g);
    shift = c->modf;
    scale = c->modf + D;
  }
  if (d.d_out <= 64 && d.head != SGD_HEAD_LOGITS) {
    // small heads normalise each fp32 row in the kernel that applies W_head
    HeadParams hp{};
    hp.h = c->h;
    hp.ldx = D;
    hp.norm_kind = d.head == SGD_HEAD_ADALN_LINEAR ? SGD_NORM_LN_PLAIN
                                                   : (d.norm == SGD_NORM_RMS ? SGD_NORM_RMS : SGD_NORM_LN);
    hp.g = d.head == SGD_HEAD_ADALN_LINEAR ? nullptr : B16(c->w.normf_w);
    hp.b = d.head == SGD_HEAD_ADALN_LINEAR || d.norm == SGD_NORM_RMS ? nullptr : B16(c->w.normf_b);
    hp.shift = shift;
    hp.scale = scale;
    hp.ld_mod = 2 * D;
    hp.eps = d.eps;
    hp.W = B16(c->w.w_head);
    hp.N = d.d_out;
    hp.K = D;
    hp.batch = d.batch;
    hp.n_tokens = d.n_tokens;
    hp.n_prefix = d.n_prefix;
    hp.out_channels = d.out_channels;
    hp.slot = c->slot;
    Op op;
    op.name = "head.linear";
    op.kernel = SGD_KERNEL_SMALL;
    op.flops = 2.0 * M * d.out_channels * D;
    op.bytes = 4.0 * M * D + 4.0 * M * d.out_channels;
    op.run = [hp](cudaStream_t s) { return head_small_launch(hp, s); };
    ops.push_back(std::move(op));
    return SGD_OK;
  }
  const int head_norm = d.norm == SGD_NORM_RMS ? SGD_NORM_RMS : SGD_NORM_LN;
  EpiParams e = epi_base(d.head == SGD_HEAD_LOGITS ? SGD_EPI_F16 : SGD_EPI_F32);
  e.out_slot = out_slot;
  e.ldo = d.head == SGD_HEAD_LOGITS ? d.d_out : d.out_channels;
  if (c->fold) {
    set_folded_norm(c, e, head_norm);
    return make_gemm_op(c, ops, "head.linear", c->h16, D, c->pw_head, D, M, d.d_out, D, e);
  }
  make_norm_op(c, ops, "head.norm", head_norm, c->w.normf_w, c->w.normf_b, nullptr, nullptr, 0);
  return make_gemm_op(c, ops, "head.linear", c->xn, D, c->pw_head, D, M, d.d_out, D, e);
}

// Stream-K workspace for the GEMM plans built so far (tickets zeroed once; every launch
// that completes leaves them zero).
int ensure_sk_ws(sgd_ctx* c) {
  int rc;
  if (c->sk_need_floats > c->sk_ws_floats) {
    if ((rc = c->alloc(&c->sk_ws, c->sk_need_floats, &c->ws_bytes))) return rc;
    c->sk_ws_floats = c->sk_need_floats;
  }
  if (c->sk_need_cnt > c->sk_cnt_n) {
    if ((rc = c->alloc(&c->sk_cnt, static_cast<size_t>(c->sk_need_cnt), &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemset(c->sk_cnt, 0, sizeof(int) * c->sk_need_cnt));
    c->sk_cnt_n = c->sk_need_cnt;
  }
  return SGD_OK;
}

// Launch a program's ops in order on `s`; with `pdl`, each kernel may begin launching while
// the one before finishes (programmatic dependent launch; every kernel waits for its
// predecessor's results before touching global memory).
int run_ops(const std::vector<Op>& ops, cudaStream_t s, bool pdl) {
  struct Scope {
    bool prev;
    explicit Scope(bool on) : prev(pdl_flag()) { pdl_flag() = on; }
    ~Scope() { pdl_flag() = prev; }
  } scope(pdl);
  for (const Op& op : ops) {
    cudaError_t e = op.run(s);
    if (e != cudaSuccess) return fail(SGD_ERR_CUDA, op.name + ": " + cudaGetErrorString(e));
  }
  return SGD_OK;
}

int check_shape(const sgd_model_desc& d, const sgd_weights& w) {
  auto bad = [](const std::string& m) { return fail(SGD_ERR_SHAPE, m); };
  if (d.n_blocks < 1 || d.n_blocks > 64) return bad("n_blocks must be in [1, 64]");
  if (d.d_head != 64 && d.d_head != 72 && d.d_head != 128) return bad("d_head must be 64, 72 or 128");
  if (d.n_heads * d.d_head != d.d) return bad("d must equal n_heads * d_head");
  if (d.d % 8 || d.d > 4096) return bad("d must be a multiple of 8 and at most 4096");
  if (d.d_ff < 8 || d.d_ff % 8) return bad("d_ff must be a positive multiple of 8");
  if (d.batch < 1 || d.n_tokens < 1 || d.batch * d.n_heads > 65535) return bad("bad batch / tokens");
  if (d.rope && d.d_head == 72) return bad("RoPE needs d_head 64 or 128");
  if (d.eps <= 0.f) return bad("eps must be > 0");
  if (d.stem < 0 || d.stem > 4 || d.block < 0 || d.block > 2 || d.norm < 0 || d.norm > 2 ||
      d.mlp < 0 || d.mlp > 3 || d.head < 0 || d.head > 3)
    return fail(SGD_ERR_ARG, "enum out of range");
  switch (d.stem) {
    case SGD_STEM_TIME_ADD:
    case SGD_STEM_IDENTITY:
      if (d.d_in != d.d || d.n_prefix) return bad("time_add / identity stems need d_in == d, no prefix");
      break;
    case SGD_STEM_PATCH:
      if (d.d_in < 1 || d.n_prefix || !w.w_stem || !w.pos_emb) return bad("patch stem needs w_stem, pos_emb");
      break;
    case SGD_STEM_PATCH_TOKENS:
      if (d.d_in < 1 || d.n_prefix != 2 || !w.w_stem || !w.pos_emb || !w.class_emb || d.n_classes < 1)
        return bad("patch-token stem needs n_prefix 2, w_stem, pos_emb, class_emb");
      break;
    case SGD_STEM_EMBED:
      if (d.vocab < 1 || !w.embed || d.n_prefix) return bad("embed stem needs vocab and embed");
      break;
  }
  if (d.block == SGD_BLOCK_ADALN) {
    if (!w.w_t1 || !w.w_t2 || !w.class_emb || d.t_freq < 8 || d.t_freq % 8 || d.batch > 16 ||
        d.norm != SGD_NORM_LN_PLAIN)
      return bad("AdaLN blocks need w_t1, w_t2, class_emb, t_freq % 8 == 0, batch <= 16, LN_PLAIN");
  }
  if (d.block == SGD_BLOCK_XATTN && (d.ctx_len < 1 || d.d_ctx < 8 || d.d_ctx % 8))
    return bad("cross-attention needs ctx_len >= 1 and d_ctx a multiple of 8");
  if (d.n_skips && (d.n_blocks != 2 * d.n_skips + 1 || !w.skip_w))
    return bad("long skips need n_blocks = 2 n_skips + 1 and skip weights");
  switch (d.head) {
    case SGD_HEAD_LINEAR:
      if (!w.w_head || !w.normf_w) return bad("linear head needs normf_w and w_head");
      if (d.d_out > 64 && (d.n_prefix || d.out_channels != d.d_out || d.d_out % 8))
        return bad("wide linear head needs out_channels == d_out (multiple of 8) and no prefix");
      if (d.out_channels > d.d_out) return bad("out_channels > d_out");
      break;
    case SGD_HEAD_ADALN_LINEAR:
      if (d.block != SGD_BLOCK_ADALN || !w.w_modf || !w.w_head || d.d_out > 64 ||
          d.out_channels > d.d_out)
        return bad("AdaLN head needs AdaLN blocks, w_modf, w_head, d_out <= 64");
      break;
    case SGD_HEAD_IDENTITY:
      if (d.n_prefix || d.out_channels != d.d) return bad("identity head needs out_channels == d");
      break;
    case SGD_HEAD_LOGITS:
      if (!w.w_head || !w.normf_w || d.d_out % 8 || d.d_out < 8) return bad("logits head needs normf_w, w_head, d_out % 8 == 0");
      break;
  }
  if (!w.blocks) return fail(SGD_ERR_ARG, "null block weights");
  // every weight is read with 8- or 16-byte vector loads
  {
    const void* top[] = {w.w_stem, w.pos_emb, w.w_t1, w.w_t2, w.class_emb, w.normf_w,
                         w.normf_b, w.w_modf, w.w_head, w.embed};
    for (const void* p : top)
      if (p && !al16(p)) return fail(SGD_ERR_ARG, "misaligned weight (16-byte alignment needed)");
    for (int i = 0; w.skip_w && i < d.n_skips; ++i)
      if (w.skip_w[i] && !al16(w.skip_w[i])) return fail(SGD_ERR_ARG, "misaligned skip weight");
  }
  for (int b = 0; b < d.n_blocks; ++b) {
    const sgd_block_weights& W = w.blocks[b];
    const void* all[] = {W.norm1_w, W.norm1_b, W.normx_w, W.normx_b, W.wx_q, W.wx_o, W.norm2_w, W.norm2_b};
    for (const void* p : all)
      if (p && !al16(p)) return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": misaligned weight");
    const void* need[] = {W.w_qkv, W.w_o, W.w_1, W.w_2};
    for (const void* p : need)
      if (!p || !al16(p)) return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": missing or misaligned weight");
    if (d.norm != SGD_NORM_LN_PLAIN && (!W.norm1_w || !W.norm2_w))
      return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": missing norm gains");
    if (d.norm == SGD_NORM_LN && (!W.norm1_b || !W.norm2_b))
      return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": missing norm shifts");
    if (d.block == SGD_BLOCK_ADALN && (!W.w_mod || !al16(W.w_mod)))
      return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": missing w_mod");
    if (d.block == SGD_BLOCK_XATTN &&
        (!W.wx_q || !W.wx_kv || !W.wx_o || !W.normx_w || !W.normx_b || !al16(W.wx_kv)))
      return fail(SGD_ERR_ARG, "block " + std::to_string(b) + ": missing cross-attention weights");
  }
  return SGD_OK;
}

int ensure_alloc(sgd_ctx* c) {
  const sgd_model_desc& d = c->d;
  const size_t M = c->M, D = d.d, F = d.d_ff;
  int rc;
  if ((rc = c->alloc(&c->h, M * D, &c->ws_bytes))) return rc;
  if ((rc = c->alloc(&c->xn, M * D, &c->ws_bytes))) return rc;
  // d_head 72 on tcgen05: heads padded to 80 columns in qkv, the gaps zero (never written)
  c->head_stride = (d.d_head == 72 && c->attn_impl == 0) ? 80 : d.d_head;
  const size_t QW = static_cast<size_t>(d.n_heads) * c->head_stride;
  if ((rc = c->alloc(&c->qkv, M * 3 * QW, &c->ws_bytes))) return rc;
  CUDA_TRY(cudaMemset(c->qkv, 0, M * 3 * QW * sizeof(f16)));
  if ((rc = c->alloc(&c->attn, M * D, &c->ws_bytes))) return rc;
  if ((rc = c->alloc(&c->act, M * F, &c->ws_bytes))) return rc;
  if ((rc = c->alloc(&c->slot, 1, &c->ws_bytes))) return rc;
  CUDA_TRY(cudaMemset(c->slot, 0, sizeof(IoSlot)));
  if (c->fold) {
    if ((rc = c->alloc(&c->h16, M * D, &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->rstat, 2 * static_cast<size_t>(kStatSlots) * M, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemset(c->rstat, 0, 2 * sizeof(float) * kStatSlots * M));
    if ((rc = c->alloc(&c->rstat_final, 2 * static_cast<size_t>(kStatSlots) * M, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemset(c->rstat_final, 0, 2 * sizeof(float) * kStatSlots * M));
    const size_t blocks = (M + 127) / 128;
    if ((rc = c->alloc(&c->stat_cnt, blocks, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemset(c->stat_cnt, 0, blocks * sizeof(int)));
  }
  if (d.block == SGD_BLOCK_ADALN) {
    if ((rc = c->alloc(&c->t_hidden, D, &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->cond_c, d.batch * D, &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->cond_silu, d.batch * D, &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->mod, static_cast<size_t>(d.n_blocks) * d.batch * 6 * D, &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->modf, d.batch * 2 * D, &c->ws_bytes))) return rc;
  }
  if (d.block == SGD_BLOCK_XATTN) {
    if ((rc = c->alloc(&c->ctx16, static_cast<size_t>(d.batch) * d.ctx_len * d.d_ctx, &c->ws_bytes))) return rc;
    c->ctxkv.assign(d.n_blocks, nullptr);
    for (int b = 0; b < d.n_blocks; ++b)
      if ((rc = c->alloc(&c->ctxkv[b], static_cast<size_t>(d.batch) * d.ctx_len * 2 * D, &c->ws_bytes))) return rc;
  }
  if (d.n_skips) {
    c->skipcat.assign(d.n_skips, nullptr);
    for (int j = 0; j < d.n_skips; ++j)
      if ((rc = c->alloc(&c->skipcat[j], M * 2 * D, &c->ws_bytes))) return rc;
  }
  if (d.rope) {
    const int half = d.d_head / 2;
    std::vector<float> cs(static_cast<size_t>(d.n_tokens) * half), sn(cs.size());
    for (int p = 0; p < d.n_tokens; ++p)
      for (int i = 0; i < half; ++i) {
        const double f = std::pow(static_cast<double>(d.rope_theta), -2.0 * i / d.d_head);
        cs[static_cast<size_t>(p) * half + i] = static_cast<float>(std::cos(p * f));
        sn[static_cast<size_t>(p) * half + i] = static_cast<float>(std::sin(p * f));
      }
    if ((rc = c->alloc(&c->rope_cos, cs.size(), &c->ws_bytes))) return rc;
    if ((rc = c->alloc(&c->rope_sin, sn.size(), &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemcpy(c->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice));
    CUDA_TRY(cudaMemcpy(c->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice));
  }
  c->cache.assign(c->U, nullptr);
  return SGD_OK;
}

// fp16 copy of a bf16 [rows, cols] weight, scaled by the largest power of two that
// keeps max |w| finite in fp16 (exact conversion of every entry in the normal range).
int prep_weight(sgd_ctx* c, const void* src, int64_t n, PW& out) {
  f16* dst = nullptr;
  int rc = c->alloc(&dst, static_cast<size_t>(n), &c->weight_bytes);
  if (rc) return rc;
  CUDA_TRY(cudaMemset(c->absmax, 0, sizeof(float)));
  CUDA_TRY(absmax_bf16_launch(B16(src), n, c->absmax, 0));
  float m = 0.f;
  CUDA_TRY(cudaMemcpy(&m, c->absmax, sizeof(float), cudaMemcpyDeviceToHost));
  int shift = 0;
  if (m > 0.f && std::isfinite(m)) {
    shift = static_cast<int>(std::floor(std::log2(65504.0 / m)));
    shift = std::max(-100, std::min(100, shift));
  }
  CUDA_TRY(convert_bf16_f16_launch(B16(src), dst, n, shift, 0));
  out.w = dst;
  out.alpha = std::ldexp(1.0f, -shift);
  return SGD_OK;
}

// The same for a weight that consumes a folded pre-norm: fp16(W diag(g) 2^shift) and, for
// LayerNorm, the column vectors alpha sum_k W'[j, k] (from the fp16 copy, so that it matches
// what the tensor cores multiply) and sum_k b_k W[j, k].
int prep_weight_folded(sgd_ctx* c, const void* src, int64_t rows, int K, const void* g, const void* b,
                       bool ln, PW& out) {
  f16* dst = nullptr;
  int rc = c->alloc(&dst, static_cast<size_t>(rows) * K, &c->weight_bytes);
  if (rc) return rc;
  CUDA_TRY(cudaMemset(c->absmax, 0, sizeof(float)));
  CUDA_TRY(absmax_scaled_launch(B16(src), B16(g), rows, K, c->absmax, 0));
  float m = 0.f;
  CUDA_TRY(cudaMemcpy(&m, c->absmax, sizeof(float), cudaMemcpyDeviceToHost));
  int shift = 0;
  if (m > 0.f && std::isfinite(m)) {
    shift = static_cast<int>(std::floor(std::log2(65504.0 / m)));
    shift = std::max(-100, std::min(100, shift));
  }
  CUDA_TRY(convert_scaled_launch(B16(src), B16(g), dst, rows, K, shift, 0));
  out.w = dst;
  out.alpha = std::ldexp(1.0f, -shift);
  if (ln) {
    float* cs = nullptr;
    float* cb = nullptr;
    const size_t padded = static_cast<size_t>(rows) + 512;
    if ((rc = c->alloc(&cs, padded, &c->weight_bytes)) || (rc = c->alloc(&cb, padded, &c->weight_bytes)))
      return rc;
    CUDA_TRY(cudaMemset(cs, 0, padded * sizeof(float)));
    CUDA_TRY(cudaMemset(cb, 0, padded * sizeof(float)));
    CUDA_TRY(rowsum_f16_launch(dst, rows, K, out.alpha, cs, 0));
    CUDA_TRY(rowdot_bf16_launch(B16(src), B16(b), rows, K, cb, 0));
    out.colsum = cs;
    out.colbias = cb;
  }
  return SGD_OK;
}

int prep_weights(sgd_ctx* c) {
  const sgd_model_desc& d = c->d;
  const int64_t D = d.d, F = d.d_ff;
  const bool gated = d.mlp == SGD_MLP_SWIGLU || d.mlp == SGD_MLP_GEGLU;
  int rc;
  if ((rc = c->alloc(&c->absmax, 1, &c->ws_bytes))) return rc;
  c->pw.assign(d.n_blocks, BlockPW{});
  for (int b = 0; b < d.n_blocks; ++b) {
    const sgd_block_weights& W = c->blk[b];
    BlockPW& P = c->pw[b];
    const bool ln = d.norm == SGD_NORM_LN;
    if (c->fold) {
      if ((rc = prep_weight_folded(c, W.w_qkv, 3 * D, D, W.norm1_w, W.norm1_b, ln, P.qkv)) ||
          (rc = prep_weight_folded(c, W.w_1, (gated ? 2 : 1) * F, D, W.norm2_w, W.norm2_b, ln, P.w1)))
        return rc;
    } else if ((rc = prep_weight(c, W.w_qkv, 3 * D * D, P.qkv)) ||
               (rc = prep_weight(c, W.w_1, (gated ? 2 : 1) * F * D, P.w1))) {
      return rc;
    }
    if ((rc = prep_weight(c, W.w_o, D * D, P.o))) return rc;
    if ((rc = prep_weight(c, W.w_2, D * F, P.w2))) return rc;
    if (d.block == SGD_BLOCK_XATTN) {
      if (c->fold)
        rc = prep_weight_folded(c, W.wx_q, D, D, W.normx_w, W.normx_b, true, P.xq);
      else
        rc = prep_weight(c, W.wx_q, D * D, P.xq);
      if (rc) return rc;
      if ((rc = prep_weight(c, W.wx_kv, 2 * D * d.d_ctx, P.xkv))) return rc;
      if ((rc = prep_weight(c, W.wx_o, D * D, P.xo))) return rc;
    }
  }
  c->pw_skip.assign(d.n_skips, PW{});
  for (int j = 0; j < d.n_skips; ++j)
    if ((rc = prep_weight(c, c->skip_w[j], D * 2 * D, c->pw_skip[j]))) return rc;
  const bool tc_head = d.head == SGD_HEAD_LOGITS || (d.head == SGD_HEAD_LINEAR && d.d_out > 64);
  if (tc_head) {
    if (c->fold)
      rc = prep_weight_folded(c, c->w.w_head, d.d_out, static_cast<int>(D), c->w.normf_w, c->w.normf_b,
                              d.norm == SGD_NORM_LN, c->pw_head);
    else
      rc = prep_weight(c, c->w.w_head, static_cast<int64_t>(d.d_out) * D, c->pw_head);
    if (rc) return rc;
  }
  CUDA_TRY(cudaDeviceSynchronize());
  return SGD_OK;
}

void drop_graphs(sgd_ctx* c) {
  for (auto e : c->execs) cudaGraphExecDestroy(e);
  for (auto g : c->graphs) cudaGraphDestroy(g);
  c->execs.clear();
  c->graphs.clear();
  c->programs.clear();
  c->drift_graph_of.clear();
  c->drift_eager.clear();
  c->scheduled = false;
}

// Cross-attention K/V of the (constant) context, projected at step 1 of a trajectory.
int ctx_kv_ops(sgd_ctx* c, const void* ctx_dev, std::vector<Op>& ops) {
  const sgd_model_desc& d = c->d;
  ops.clear();
  for (int b = 0; b < d.n_blocks; ++b) {
    EpiParams e = epi_base(SGD_EPI_F16);
    e.out = c->ctxkv[b];
    e.ldo = 2 * d.d;
    int rc = make_gemm_op(c, ops, "b" + std::to_string(b) + ".xattn.ctx_kv", c->ctx16, d.d_ctx,
                          c->pw[b].xkv, d.d_ctx, d.batch * d.ctx_len, 2 * d.d, d.d_ctx, e);
    if (rc) return rc;
  }
  return SGD_OK;
}

int check_step_args(sgd_ctx* c, const void* in, void* out, const sgd_cond* cond, int step) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (!c->scheduled) return fail(SGD_ERR_STATE, "no schedule installed");
  if (!in || !out) return fail(SGD_ERR_ARG, "null state or output");
  if (step < 1 || step > c->T) return fail(SGD_ERR_ARG, "step outside [1, T]");
  if (step != 1 && step != c->last_step + 1)
    return fail(SGD_ERR_CACHE_INVALID, "step " + std::to_string(step) + " after step " +
                                           std::to_string(c->last_step) +
                                           ": caches need steps 1..s-1 since the last reset");
  if ((c->d.n_classes && c->d.block == SGD_BLOCK_ADALN) || c->d.stem == SGD_STEM_PATCH_TOKENS) {
    if (!cond || !cond->class_ids) return fail(SGD_ERR_ARG, "model needs class ids");
  }
  if (c->d.block == SGD_BLOCK_XATTN && step == 1 && (!cond || !cond->ctx))
    return fail(SGD_ERR_ARG, "cross-attention model needs a context at step 1");
  if (!al16(in) || !al16(out)) return fail(SGD_ERR_ARG, "state/output must be 16-byte aligned");
  return SGD_OK;
}

int prepare_step(sgd_ctx* c, const void* in, void* out, float t, const sgd_cond* cond, int step,
                 cudaStream_t s) {
  IoSlot v{};
  v.state = in;
  v.out = out;
  v.class_ids = cond ? cond->class_ids : nullptr;
  v.ctx = cond ? cond->ctx : nullptr;
  v.t = t;
  v.step = step;
  CUDA_TRY(io_set_launch(c->slot, v, s));
  if (step == 1 && c->d.block == SGD_BLOCK_XATTN) {
    const int64_t n = static_cast<int64_t>(c->d.batch) * c->d.ctx_len * c->d.d_ctx;
    CUDA_TRY(convert_bf16_f16_launch(B16(cond->ctx), c->ctx16, n, 0, s));
    std::vector<Op> ops;
    int rc = ctx_kv_ops(c, cond->ctx, ops);
    if (rc) return rc;
    if ((rc = ensure_sk_ws(c)) || (rc = run_ops(ops, s, c->pdl))) return rc;
  }
  return SGD_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" {

const char* sgd_last_error(void) { return g_err.c_str(); }

int sgd_create(const sgd_model_desc* desc, const sgd_weights* w, sgd_ctx** out) {
  if (!desc || !w || !out) return fail(SGD_ERR_ARG, "null argument");
  *out = nullptr;
  if (desc->flags & ~(SGD_FLAG_SIMT_GEMM | SGD_FLAG_MMA_SYNC_ATTENTION | SGD_FLAG_GEMM_BK64 | SGD_FLAG_PDL |
                      SGD_FLAG_FOLD_NORM))
    return fail(SGD_ERR_ARG, "unknown flag bits");
  int rc = check_shape(*desc, *w);
  if (rc) return rc;
  auto* c = new (std::nothrow) sgd_ctx();
  if (!c) return fail(SGD_ERR_OOM, "host allocation failed");
  c->d = *desc;
  c->blk.assign(w->blocks, w->blocks + desc->n_blocks);
  c->w = *w;
  c->w.blocks = c->blk.data();
  for (int j = 0; j < desc->n_skips; ++j) c->skip_w.push_back(B16(w->skip_w[j]));
  c->w.skip_w = nullptr;
  if (cudaGetDevice(&c->device) != cudaSuccess) {
    delete c;
    return fail(SGD_ERR_CUDA, "no CUDA device");
  }
  c->M = desc->batch * desc->n_tokens;
  c->attn_impl = (desc->flags & SGD_FLAG_MMA_SYNC_ATTENTION) ? 1 : 0;
  c->pdl = (desc->flags & SGD_FLAG_PDL) != 0;
  // RMSNorm / LayerNorm pre-norms fold into the GEMMs that follow them on request; the AdaLN
  // modulation (a per-sample scale of the weight's columns) and the SIMT debug GEMM do not
  c->fold = (desc->norm == SGD_NORM_RMS || desc->norm == SGD_NORM_LN) &&
            (desc->flags & SGD_FLAG_FOLD_NORM) && !(desc->flags & SGD_FLAG_SIMT_GEMM);
  c->nbr = desc->block == SGD_BLOCK_XATTN ? 3 : 2;
  c->U = desc->n_blocks * c->nbr;
  if ((rc = ensure_alloc(c)) || (rc = prep_weights(c))) {
    delete c;
    return rc;
  }
  if (cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
    delete c;
    return fail(SGD_ERR_CUDA, "stream creation failed");
  }
  *out = c;
  g_err.clear();
  return SGD_OK;
}

int sgd_compile_schedule(int T, int n_units, const int32_t* lifetimes, const int32_t* groups,
                         int32_t* pattern_of_step, int32_t* writes_at_step, int32_t* n_patterns) {
  int rc = validate_schedule(T, n_units, lifetimes, groups, -1);
  if (rc) return rc;
  std::vector<int> pos, wr;
  std::vector<std::vector<uint8_t>> pats;
  compile_patterns(T, n_units, lifetimes, pos, wr, pats);
  for (int s = 0; s < T; ++s) {
    if (pattern_of_step) pattern_of_step[s] = pos[s];
    if (writes_at_step) writes_at_step[s] = wr[s];
  }
  if (n_patterns) *n_patterns = static_cast<int32_t>(pats.size());
  return SGD_OK;
}

// Capture `ops` into a graph; the program, graph and executable are kept in the context.
static int capture_program(sgd_ctx* c, std::vector<Op>&& ops, int* gid) {
  cudaGraph_t g = nullptr;
  CUDA_TRY(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeRelaxed));
  int rc = run_ops(ops, c->cap_stream, c->pdl);
  cudaError_t ce = cudaStreamEndCapture(c->cap_stream, &g);
  if (rc) {
    if (g) cudaGraphDestroy(g);
    return rc;
  }
  if (ce != cudaSuccess) return fail(SGD_ERR_CUDA, std::string("graph capture: ") + cudaGetErrorString(ce));
  cudaGraphExec_t ex = nullptr;
  ce = cudaGraphInstantiate(&ex, g, 0);
  if (ce != cudaSuccess) {
    cudaGraphDestroy(g);
    return fail(SGD_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(ce));
  }
  *gid = static_cast<int>(c->graphs.size());
  c->graphs.push_back(g);
  c->execs.push_back(ex);
  c->programs.push_back(std::move(ops));
  return SGD_OK;
}

// Buffers of the drift policy: every unit's cache (any active step may be a unit's last),
// the per-group input snapshots, partial and final drift sums, and their host copy.
static int ensure_drift_buffers(sgd_ctx* c) {
  int rc;
  for (int u = 0; u < c->U; ++u)
    if (!c->cache[u] && (rc = c->alloc(&c->cache[u], static_cast<size_t>(c->M) * c->d.d, &c->cache_bytes)))
      return rc;
  const size_t G = static_cast<size_t>(c->n_groups);
  if (c->drift_alloc_groups < G) {
    const size_t n = static_cast<size_t>(c->M) * c->d.d;
    if ((rc = c->alloc(&c->snap, G * n, &c->ws_bytes)) ||
        (rc = c->alloc(&c->drift_part, G * 2 * kDriftBlocks, &c->ws_bytes)) ||
        (rc = c->alloc(&c->drift_sums, G * 2, &c->ws_bytes)))
      return rc;
    CUDA_TRY(cudaMemset(c->snap, 0, G * n * sizeof(float)));
    if (c->drift_host) cudaFreeHost(c->drift_host);
    c->drift_host = nullptr;
    CUDA_TRY(cudaHostAlloc(reinterpret_cast<void**>(&c->drift_host), G * 2 * sizeof(double), cudaHostAllocDefault));
    c->drift_alloc_groups = G;
  }
  if (!c->ev_drift) CUDA_TRY(cudaEventCreateWithFlags(&c->ev_drift, cudaEventDisableTiming));
  return SGD_OK;
}

static int build_graphs(sgd_ctx* c) {
  const int T = c->T;
  int rc;
  drop_graphs(c);
  if (c->policy == SGD_POLICY_DRIFT) {
    // the graph library: one graph per active set of the static schedule, in which every
    // active unit stores its update and every group's drift is reduced
    if ((rc = ensure_drift_buffers(c))) return rc;
    for (const auto& pat : c->patterns) {
      std::vector<Op> ops;
      if ((rc = build_program(c, pat, pat, ops)) || (rc = ensure_sk_ws(c))) return rc;
      int gid = -1;
      if ((rc = capture_program(c, std::move(ops), &gid))) return rc;
      c->drift_graph_of[pat] = gid;
    }
    c->graph_of_step.assign(T + 1, -1);
    c->drift_used.assign(T + 1, {});
    c->mask_used.assign(T + 1, {});
    c->last_step = 0;
    c->scheduled = true;
    return SGD_OK;
  }
  // graph variants: (pattern, cache-store set); the store set is non-empty only at steps
  // s = S_u < T, so each such step gets its own variant.
  std::map<std::pair<int, int>, int> key_to_graph;
  c->graph_of_step.assign(T + 1, -1);
  for (int s = 1; s <= T; ++s) {
    const int pid = c->pattern_of_step[s - 1];
    const int key2 = c->writes[s - 1] ? s : -1;
    auto it = key_to_graph.find({pid, key2});
    if (it != key_to_graph.end()) {
      c->graph_of_step[s] = it->second;
      continue;
    }
    std::vector<uint8_t> write(c->U, 0);
    for (int u = 0; u < c->U; ++u) write[u] = (c->S[u] == s && s < T) ? 1 : 0;
    std::vector<Op> ops;
    if ((rc = build_program(c, c->patterns[pid], write, ops)) || (rc = ensure_sk_ws(c))) return rc;
    int gid = -1;
    if ((rc = capture_program(c, std::move(ops), &gid))) return rc;
    key_to_graph[{pid, key2}] = gid;
    c->graph_of_step[s] = gid;
  }
  c->last_step = 0;
  c->scheduled = true;
  return SGD_OK;
}

int sgd_set_schedule(sgd_ctx* c, int T, int n_units, const int32_t* lifetimes, const int32_t* groups) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  int rc = validate_schedule(T, n_units, lifetimes, groups, c->U);
  if (rc) return rc;
  CUDA_TRY(cudaSetDevice(c->device));
  drop_graphs(c);
  c->T = T;
  c->S.assign(lifetimes, lifetimes + n_units);
  c->groups.assign(groups, groups + n_units);
  compile_patterns(T, n_units, lifetimes, c->pattern_of_step, c->writes, c->patterns);
  // groups numbered by their first unit; the static schedule's active-group count per step
  {
    std::map<int32_t, int> index;
    c->group_of_unit.assign(n_units, 0);
    c->group_start.assign(n_units, 0);
    std::vector<int32_t> life;
    for (int u = 0; u < n_units; ++u) {
      auto it = index.find(groups[u]);
      if (it == index.end()) {
        const int g = static_cast<int>(index.size());
        index[groups[u]] = g;
        c->group_start[u] = 1;
        life.push_back(lifetimes[u]);
        c->group_of_unit[u] = g;
      } else {
        c->group_of_unit[u] = it->second;
      }
    }
    c->n_groups = static_cast<int>(index.size());
    c->m_of_step.assign(T + 1, 0);
    for (int s = 1; s <= T; ++s)
      for (int32_t l : life) c->m_of_step[s] += l >= s ? 1 : 0;
  }
  // caches only for units that are ever frozen
  for (int u = 0; u < c->U; ++u)
    if (c->S[u] < T && !c->cache[u]) {
      if ((rc = c->alloc(&c->cache[u], static_cast<size_t>(c->M) * c->d.d, &c->cache_bytes))) return rc;
    }
  if ((rc = build_graphs(c))) return rc;
  g_err.clear();
  return SGD_OK;
}

int sgd_set_exec_mode(sgd_ctx* c, int mode) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (mode < SGD_EXEC_JAGGED_GRAPH || mode > SGD_EXEC_PADDED_GRAPH)
    return fail(SGD_ERR_ARG, "unknown execution mode");
  if (mode == SGD_EXEC_PADDED_GRAPH && c->policy == SGD_POLICY_DRIFT)
    return fail(SGD_ERR_STATE, "the drift policy runs with jagged graphs or eagerly, not padded graphs");
  int rc;
  if (mode == SGD_EXEC_PADDED_GRAPH && !c->h_pad &&
      (rc = c->alloc(&c->h_pad, static_cast<size_t>(c->M) * c->d.d, &c->ws_bytes)))
    return rc;
  const bool rebuild = (mode == SGD_EXEC_PADDED_GRAPH) != (c->exec_mode == SGD_EXEC_PADDED_GRAPH);
  c->exec_mode = mode;
  if (rebuild && c->scheduled) {
    CUDA_TRY(cudaSetDevice(c->device));
    if ((rc = build_graphs(c))) return rc;
  }
  c->last_step = 0;
  return SGD_OK;
}

int sgd_set_policy(sgd_ctx* c, int policy) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (policy != SGD_POLICY_STATIC && policy != SGD_POLICY_DRIFT) return fail(SGD_ERR_ARG, "unknown policy");
  if (policy == SGD_POLICY_DRIFT && c->exec_mode == SGD_EXEC_PADDED_GRAPH)
    return fail(SGD_ERR_STATE, "the drift policy runs with jagged graphs or eagerly, not padded graphs");
  const bool rebuild = policy != c->policy;
  c->policy = policy;
  if (rebuild && c->scheduled) {
    CUDA_TRY(cudaSetDevice(c->device));
    int rc;
    if ((rc = build_graphs(c))) return rc;
  }
  c->last_step = 0;
  return SGD_OK;
}

namespace {

// App. B.1 routing for step `step`: the active groups (step 1 all, step 2 the m_2 lowest,
// later the m_s with the largest lagged drift of step - 1, ties to the lower index),
// recorded with the drifts they were ranked by; returns the unit mask.
int drift_route(sgd_ctx* c, int step, std::vector<uint8_t>& mask) {
  const int G = c->n_groups;
  const int m = c->m_of_step[step];
  if (step == 1) {  // a new trajectory: forget the previous one's records
    for (auto& v : c->drift_used) v.clear();
    for (auto& v : c->mask_used) v.clear();
  }
  std::vector<double> dv(G, 0.0);
  std::vector<int> order(G);
  for (int g = 0; g < G; ++g) order[g] = g;
  if (step >= 3) {
    CUDA_TRY(cudaEventSynchronize(c->ev_drift));  // step - 1's sums are on the host
    for (int g = 0; g < G; ++g)
      dv[g] = std::sqrt(c->drift_host[2 * g]) / (std::sqrt(c->drift_host[2 * g + 1]) + 1e-8);
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return dv[a] > dv[b]; });
  }
  std::vector<uint8_t> on(G, 0);
  for (int i = 0; i < (step == 1 ? G : m); ++i) on[order[i]] = 1;
  mask.assign(c->U, 0);
  for (int u = 0; u < c->U; ++u) mask[u] = on[c->group_of_unit[u]];
  c->drift_used[step] = dv;
  c->mask_used[step] = mask;
  return SGD_OK;
}

// One step under the drift policy: route, replay the library graph of the chosen active set
// or run its op list eagerly, then queue the copy of this step's drift sums to the host.
int drift_step(sgd_ctx* c, int step, cudaStream_t s) {
  std::vector<uint8_t> mask;
  int rc;
  if ((rc = drift_route(c, step, mask))) return rc;
  auto it = c->drift_graph_of.find(mask);
  if (it != c->drift_graph_of.end() && c->exec_mode == SGD_EXEC_JAGGED_GRAPH) {
    CUDA_TRY(cudaGraphLaunch(c->execs[it->second], s));
    ++c->graph_steps;
  } else {
    if (it != c->drift_graph_of.end()) {
      if ((rc = run_ops(c->programs[it->second], s, c->pdl))) return rc;
    } else {
      auto e = c->drift_eager.find(mask);
      if (e == c->drift_eager.end()) {
        std::vector<Op> ops;
        if ((rc = build_program(c, mask, mask, ops)) || (rc = ensure_sk_ws(c))) return rc;
        e = c->drift_eager.emplace(mask, std::move(ops)).first;
      }
      if ((rc = run_ops(e->second, s, c->pdl))) return rc;
    }
    ++c->eager_steps;
  }
  CUDA_TRY(cudaMemcpyAsync(c->drift_host, c->drift_sums, sizeof(double) * 2 * c->n_groups,
                           cudaMemcpyDeviceToHost, s));
  CUDA_TRY(cudaEventRecord(c->ev_drift, s));
  return SGD_OK;
}

}  // namespace

int sgd_step(sgd_ctx* c, const void* in, void* out, float t, const sgd_cond* cond, int step,
             void* stream) {
  int rc = check_step_args(c, in, out, cond, step);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = prepare_step(c, in, out, t, cond, step, s))) return rc;
  if (c->policy == SGD_POLICY_DRIFT) {
    if ((rc = drift_step(c, step, s))) return rc;
    c->last_step = step == c->T ? 0 : step;
    return SGD_OK;
  }
  if (c->exec_mode == SGD_EXEC_EAGER) {
    if ((rc = run_ops(c->programs[c->graph_of_step[step]], s, c->pdl))) return rc;  // one launch per op
  } else {
    CUDA_TRY(cudaGraphLaunch(c->execs[c->graph_of_step[step]], s));
  }
  c->last_step = step == c->T ? 0 : step;
  return SGD_OK;
}

int sgd_step_profile(sgd_ctx* c, const void* in, void* out, float t, const sgd_cond* cond, int step,
                     void* stream, sgd_op_record* rec, int max_rec, int* n_rec) {
  int rc = check_step_args(c, in, out, cond, step);
  if (rc) return rc;
  if (c->policy != SGD_POLICY_STATIC) return fail(SGD_ERR_STATE, "profiled steps need the static policy");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = prepare_step(c, in, out, t, cond, step, s))) return rc;
  const std::vector<Op>& ops = c->programs[c->graph_of_step[step]];
  std::vector<cudaEvent_t> ev(2 * ops.size());
  for (auto& e : ev) CUDA_TRY(cudaEventCreate(&e));
  for (size_t i = 0; i < ops.size(); ++i) {
    cudaEventRecord(ev[2 * i], s);
    cudaError_t e = ops[i].run(s);
    cudaEventRecord(ev[2 * i + 1], s);
    if (e != cudaSuccess) {
      for (auto& x : ev) cudaEventDestroy(x);
      return fail(SGD_ERR_CUDA, ops[i].name + ": " + cudaGetErrorString(e));
    }
  }
  cudaError_t se = cudaStreamSynchronize(s);
  int n = 0;
  for (size_t i = 0; i < ops.size() && static_cast<int>(i) < max_rec; ++i, ++n) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, ev[2 * i], ev[2 * i + 1]);
    if (rec) {
      memset(&rec[i], 0, sizeof(sgd_op_record));
      strncpy(rec[i].name, ops[i].name.c_str(), sizeof(rec[i].name) - 1);
      rec[i].kernel = ops[i].kernel;
      rec[i].ms = ms;
      rec[i].flops = ops[i].flops;
      rec[i].bytes = ops[i].bytes;
    }
  }
  for (auto& x : ev) cudaEventDestroy(x);
  if (n_rec) *n_rec = n;
  if (se != cudaSuccess) return fail(SGD_ERR_CUDA, std::string("profile sync: ") + cudaGetErrorString(se));
  c->last_step = step == c->T ? 0 : step;
  return SGD_OK;
}

int sgd_step_host(sgd_ctx* c, const void* in_host, void* out_host, float t, const int32_t* cls_host,
                  const void* ctx_host, int step, void* stream) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (!in_host || !out_host) return fail(SGD_ERR_ARG, "null host buffer");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int rc;
  if (!c->st_in && (rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_in), c->in_bytes(), &c->ws_bytes))) return rc;
  if (!c->st_out && (rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_out), c->out_bytes(), &c->ws_bytes))) return rc;
  sgd_cond cond{};
  if (cls_host) {
    if (!c->st_cls && (rc = c->alloc(&c->st_cls, c->d.batch, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemcpyAsync(c->st_cls, cls_host, c->d.batch * 4, cudaMemcpyHostToDevice, s));
    cond.class_ids = c->st_cls;
  }
  if (ctx_host && step == 1) {
    const size_t cb = static_cast<size_t>(c->d.batch) * c->d.ctx_len * c->d.d_ctx * 2;
    if (!c->st_ctx && (rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_ctx), cb, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemcpyAsync(c->st_ctx, ctx_host, cb, cudaMemcpyHostToDevice, s));
  }
  if (ctx_host) cond.ctx = c->st_ctx;
  CUDA_TRY(cudaMemcpyAsync(c->st_in, in_host, c->in_bytes(), cudaMemcpyHostToDevice, s));
  if ((rc = sgd_step(c, c->st_in, c->st_out, t, &cond, step, stream))) return rc;
  CUDA_TRY(cudaMemcpyAsync(out_host, c->st_out, c->out_bytes(), cudaMemcpyDeviceToHost, s));
  CUDA_TRY(cudaStreamSynchronize(s));
  return SGD_OK;
}

int sgd_step_host_async(sgd_ctx* c, const void* in_host, void* out_host, float t, const int32_t* cls_host,
                        const void* ctx_host, int step, void* stream) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (!in_host || !out_host) return fail(SGD_ERR_ARG, "null host buffer");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int rc;
  if (!c->copy_stream) {
    CUDA_TRY(cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
    for (int i = 0; i < 2; ++i) {
      CUDA_TRY(cudaEventCreateWithFlags(&c->ev_done[i], cudaEventDisableTiming));
      CUDA_TRY(cudaEventCreateWithFlags(&c->ev_copied[i], cudaEventDisableTiming));
      if ((rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_out2[i]), c->out_bytes(), &c->ws_bytes))) return rc;
    }
    CUDA_TRY(cudaEventCreateWithFlags(&c->ev_last, cudaEventDisableTiming));
    if (!c->st_in && (rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_in), c->in_bytes(), &c->ws_bytes))) return rc;
  }
  const int k = c->async_slot;
  sgd_cond cond{};
  if (cls_host) {
    if (!c->st_cls && (rc = c->alloc(&c->st_cls, c->d.batch, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemcpyAsync(c->st_cls, cls_host, c->d.batch * 4, cudaMemcpyHostToDevice, s));
    cond.class_ids = c->st_cls;
  }
  if (ctx_host && step == 1) {
    const size_t cb = static_cast<size_t>(c->d.batch) * c->d.ctx_len * c->d.d_ctx * 2;
    if (!c->st_ctx && (rc = c->alloc(reinterpret_cast<uint8_t**>(&c->st_ctx), cb, &c->ws_bytes))) return rc;
    CUDA_TRY(cudaMemcpyAsync(c->st_ctx, ctx_host, cb, cudaMemcpyHostToDevice, s));
  }
  if (ctx_host) cond.ctx = c->st_ctx;
  CUDA_TRY(cudaMemcpyAsync(c->st_in, in_host, c->in_bytes(), cudaMemcpyHostToDevice, s));
  // pinned host output (device-mapped, as cudaHostAlloc memory is under unified addressing):
  // the step's output kernel writes it directly over the host link.  A separate copy of
  // the LLaDA-shaped step's 1 GB of logits ran at ~70 GB/s beside the step's own HBM
  // traffic and left the GPU waiting for it every step.
  {
    cudaPointerAttributes pa{};
    if (cudaPointerGetAttributes(&pa, out_host) == cudaSuccess && pa.type == cudaMemoryTypeHost &&
        pa.devicePointer != nullptr) {
      if ((rc = sgd_step(c, c->st_in, pa.devicePointer, t, &cond, step, stream))) return rc;
      CUDA_TRY(cudaEventRecord(c->ev_last, s));
      c->ev_last_used = true;
      return SGD_OK;
    }
    cudaGetLastError();  // a pointer the runtime does not know (pageable memory)
  }
  // the output buffer of slot k is free once its previous copy to the host has finished
  CUDA_TRY(cudaStreamWaitEvent(s, c->ev_copied[k], 0));
  if ((rc = sgd_step(c, c->st_in, c->st_out2[k], t, &cond, step, stream))) return rc;
  CUDA_TRY(cudaEventRecord(c->ev_done[k], s));
  CUDA_TRY(cudaStreamWaitEvent(c->copy_stream, c->ev_done[k], 0));
  CUDA_TRY(cudaMemcpyAsync(out_host, c->st_out2[k], c->out_bytes(), cudaMemcpyDeviceToHost, c->copy_stream));
  CUDA_TRY(cudaEventRecord(c->ev_copied[k], c->copy_stream));
  c->async_slot ^= 1;
  return SGD_OK;
}

int sgd_host_wait(sgd_ctx* c) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  if (c->ev_last_used) CUDA_TRY(cudaEventSynchronize(c->ev_last));
  if (c->copy_stream) CUDA_TRY(cudaStreamSynchronize(c->copy_stream));
  return SGD_OK;
}

int sgd_get_active_mask(const sgd_ctx* c, int step, uint8_t* mask, int n_units) {
  if (!c || !mask) return fail(SGD_ERR_ARG, "null argument");
  if (!c->scheduled) return fail(SGD_ERR_STATE, "no schedule installed");
  if (step < 1 || step > c->T) return fail(SGD_ERR_ARG, "step outside [1, T]");
  if (n_units != c->U) return fail(SGD_ERR_ARG, "n_units mismatch");
  if (c->policy == SGD_POLICY_DRIFT) {
    if (static_cast<size_t>(step) >= c->mask_used.size() || c->mask_used[step].empty())
      return fail(SGD_ERR_STATE, "step " + std::to_string(step) + " has not run since the last reset");
    for (int u = 0; u < n_units; ++u) mask[u] = c->mask_used[step][u];
    return SGD_OK;
  }
  const auto& m = c->patterns[c->pattern_of_step[step - 1]];
  for (int u = 0; u < n_units; ++u) mask[u] = m[u];
  return SGD_OK;
}

int sgd_get_drift(const sgd_ctx* c, int step, double* drift, int n_groups) {
  if (!c || !drift) return fail(SGD_ERR_ARG, "null argument");
  if (c->policy != SGD_POLICY_DRIFT) return fail(SGD_ERR_STATE, "the static policy records no drift");
  if (!c->scheduled) return fail(SGD_ERR_STATE, "no schedule installed");
  if (step < 1 || step > c->T) return fail(SGD_ERR_ARG, "step outside [1, T]");
  if (n_groups != c->n_groups) return fail(SGD_ERR_ARG, "n_groups mismatch");
  if (static_cast<size_t>(step) >= c->drift_used.size() || c->drift_used[step].empty())
    return fail(SGD_ERR_STATE, "step " + std::to_string(step) + " has not run since the last reset");
  for (int g = 0; g < n_groups; ++g) drift[g] = c->drift_used[step][g];
  return SGD_OK;
}

int sgd_get_info(const sgd_ctx* c, sgd_info* info) {
  if (!c || !info) return fail(SGD_ERR_ARG, "null argument");
  memset(info, 0, sizeof(*info));
  info->n_units = c->U;
  info->n_patterns = static_cast<int>(c->patterns.size());
  info->n_graphs = static_cast<int>(c->graphs.size());
  info->T = c->scheduled ? c->T : 0;
  info->policy = c->policy;
  info->n_groups = c->scheduled ? c->n_groups : 0;
  info->graph_steps = c->graph_steps;
  info->eager_steps = c->eager_steps;
  int64_t ls = 0;
  if (c->scheduled)
    for (int u = 0; u < c->U; ++u) ls += c->S[u];
  info->layer_steps = ls;
  info->cache_bytes = c->cache_bytes;
  info->workspace_bytes = c->ws_bytes;
  info->weight_bytes = c->weight_bytes;
  return SGD_OK;
}

int sgd_reset(sgd_ctx* c) {
  if (!c) return fail(SGD_ERR_ARG, "null context");
  c->last_step = 0;
  for (auto& v : c->drift_used) v.clear();
  for (auto& v : c->mask_used) v.clear();
  // a GEMM that stopped on an expired wait may have left stream-K tickets behind
  if (c->sk_cnt) {
    CUDA_TRY(cudaSetDevice(c->device));
    CUDA_TRY(cudaMemset(c->sk_cnt, 0, sizeof(int) * c->sk_cnt_n));
  }
  return SGD_OK;
}

int sgd_check_device(sgd_ctx* c, void* stream) {
  (void)c;
  CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int st = 0;
  int rc = sgd_kernel_status(&st);
  if (rc) return rc;
  if (st) return fail(SGD_ERR_DEVICE_TIMEOUT, "a kernel's bounded wait expired (code " + std::to_string(st) + ")");
  int clamped = 0;
  if ((rc = sgd_kernel_f16_clamped(&clamped))) return rc;
  if (clamped)
    return fail(SGD_ERR_RANGE, "an fp16 activation or cache value was outside fp16's range "
                               "(or NaN) and was clamped to +-65504");
  return SGD_OK;
}

void sgd_destroy(sgd_ctx* c) { delete c; }

int sgd_sampler_update(float* z, const float* eps, float alpha, float beta, int64_t n, void* stream) {
  if (!z || !eps || n < 0) return fail(SGD_ERR_ARG, "bad sampler arguments");
  CUDA_TRY(sampler_launch(z, eps, alpha, beta, n, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

// ----- kernel-level entry points (include/sgd_kernels.h) -----

namespace {

// Stream-K workspace of the kernel-level GEMM entry, one per (device, stream): launches on
// one stream run in order, so they can share it.  Grown on demand (after the stream has
// finished with the old one).
struct KernelWs {
  float* ws = nullptr;
  size_t floats = 0;
  int* cnt = nullptr;
  int n_cnt = 0;
};
std::mutex g_kws_mu;
std::map<std::pair<int, void*>, KernelWs> g_kws;

int kernel_ws(int dev, void* stream, size_t floats, int n_cnt, KernelWs** out) {
  std::lock_guard<std::mutex> lk(g_kws_mu);
  KernelWs& w = g_kws[{dev, stream}];
  if (floats > w.floats || n_cnt > w.n_cnt) {
    CUDA_TRY(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
    if (floats > w.floats) {
      if (w.ws) cudaFree(w.ws);
      w.ws = nullptr;
      w.floats = 0;
      cudaError_t e = cudaMalloc(&w.ws, floats * sizeof(float));
      if (e != cudaSuccess) return fail(SGD_ERR_OOM, std::string("cudaMalloc: ") + cudaGetErrorString(e));
      w.floats = floats;
    }
    if (n_cnt > w.n_cnt) {
      if (w.cnt) cudaFree(w.cnt);
      w.cnt = nullptr;
      w.n_cnt = 0;
      cudaError_t e = cudaMalloc(&w.cnt, n_cnt * sizeof(int));
      if (e != cudaSuccess) return fail(SGD_ERR_OOM, std::string("cudaMalloc: ") + cudaGetErrorString(e));
      CUDA_TRY(cudaMemset(w.cnt, 0, n_cnt * sizeof(int)));
      w.n_cnt = n_cnt;
    }
  }
  *out = &w;
  return SGD_OK;
}

// The kernel-level GEMM arguments as a validated plan (variant codes: sgd_kernel_gemm);
// returns an sgd_status.  Nothing touches the device before the checks pass.
int kernel_gemm_plan(const void* A, int lda, const void* B, int ldb, int M, int N, int K,
                     const sgd_epilogue_args* ea, int variant, GemmPlan& p) {
  if (!ea) return fail(SGD_ERR_ARG, "null epilogue");
  if (ea->kind < 0 || ea->kind > SGD_EPI_ROPE) return fail(SGD_ERR_ARG, "bad epilogue kind");
  if (variant < 0 || variant > 12 || variant == 2 || variant == 4)
    return fail(SGD_ERR_ARG, "gemm: variant must be 0, 1, 3 or 5..12");
  p.A = H16(A);
  p.lda = lda;
  p.B = H16(B);
  p.ldb = ldb;
  p.M = M;
  p.N = N;
  p.K = K;
  p.simt = variant == 1;
  p.bk = variant == 3 ? 32 : 64;
  if (variant == 5) { p.bn = 256; p.epiw = 4; }
  if (variant == 6) { p.bn = 256; p.epiw = 8; }
  if (variant == 7) { p.bn = 128; p.epiw = 8; p.sk = 0; }
  if (variant == 8) p.sk = 0;
  if (variant == 9) p.sk = 1;
  if (variant == 10) { p.bn = 224; p.epiw = 8; }
  if (variant == 11) p.group_m = 0;
  if (variant == 12) p.group_m = 16;
  EpiParams& e = p.epi;
  e = EpiParams{};
  e.kind = ea->kind;
  e.alpha = ea->alpha != 0.f ? ea->alpha : 1.f;
  e.out = ea->out;
  e.ldo = ea->ldo;
  e.h = ea->h;
  e.ldh = ea->ldh;
  e.cache = static_cast<f16*>(ea->cache);
  e.ld_cache = ea->ld_cache;
  e.gate = ea->gate;
  e.ld_gate = ea->ld_gate;
  e.rows_per_batch = ea->rows_per_batch > 0 ? ea->rows_per_batch : 1;
  e.act = ea->act;
  e.rope_cos = ea->rope_cos;
  e.rope_sin = ea->rope_sin;
  e.rope_tokens = ea->rope_tokens;
  e.d_head = ea->d_head;
  e.rope_cols = ea->rope_cols;
  e.M = M;
  e.N = N;
  e.norm = ea->norm;
  e.rstat = ea->rstat;
  e.stat_slots = ea->stat_slots;
  e.stat_ld = ea->stat_ld;
  e.norm_eps = ea->norm_eps;
  e.norm_inv_d = 1.0f / static_cast<float>(K);
  e.colsum = ea->colsum;
  e.colbias = ea->colbias;
  e.h16 = static_cast<f16*>(ea->h16);
  e.stat_out = ea->stat_out;
  e.stat_out_ld = ea->stat_out_ld;
  e.stat_cnt = ea->stat_cnt;
  e.stat_final = ea->stat_final;
  const char* why = "";
  const int rc = gemm_plan(p, &why);
  if (rc) return fail(rc == -5 ? SGD_ERR_CUDA : (rc == -1 ? SGD_ERR_ARG : SGD_ERR_SHAPE), why);
  return SGD_OK;
}

}  // namespace

int sgd_kernel_gemm(const void* A, int lda, const void* B, int ldb, int M, int N, int K,
                    const sgd_epilogue_args* ea, int use_simt, void* stream) {
  GemmPlan p;
  const int rc = kernel_gemm_plan(A, lda, B, ldb, M, N, K, ea, use_simt, p);
  if (rc) return rc;
  if (p.sk_tiles > 0) {
    int dev = 0;
    CUDA_TRY(cudaGetDevice(&dev));
    KernelWs* w = nullptr;
    const int wrc = kernel_ws(dev, stream, gemm_ws_floats(p), p.sk_tiles, &w);
    if (wrc) return wrc;
    p.ws_ref = &w->ws;
    p.cnt_ref = &w->cnt;
    // a launch that stopped on an expired wait can leave counters behind; start from zero
    CUDA_TRY(cudaMemsetAsync(w->cnt, 0, sizeof(int) * p.sk_tiles, static_cast<cudaStream_t>(stream)));
  }
  CUDA_TRY(gemm_launch(p, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_kernel_gemm_static_ws(const void* A, int lda, const void* B, int ldb, int M, int N, int K,
                              const sgd_epilogue_args* ea, int variant, void* stream) {
  GemmPlan p;
  const int rc = kernel_gemm_plan(A, lda, B, ldb, M, N, K, ea, variant, p);
  if (rc) return rc;
  const char* why = "";
  float* ws = nullptr;
  int* tickets = nullptr;
  if (p.sk_tiles > 0) {
    size_t cap = 0;
    int n_cap = 0;
    if (gemm_static_scratch(&ws, &cap, &tickets, &n_cap, &why)) return fail(SGD_ERR_CUDA, why);
    if (gemm_ws_floats(p) > cap || p.sk_tiles > n_cap)
      return fail(SGD_ERR_SHAPE, "gemm: the stream-K split of this problem needs " +
                                     std::to_string(gemm_ws_floats(p) * sizeof(float)) +
                                     " bytes of partial tiles, more than the " + std::to_string(cap * sizeof(float)) +
                                     "-byte static scratch (use sgd_kernel_gemm, or variant 8)");
    p.ws_ref = &ws;
    p.cnt_ref = &tickets;
    // the tickets must start at zero (a launch stopped on an expired wait can leave some)
    CUDA_TRY(cudaMemsetAsync(tickets, 0, sizeof(int) * p.sk_tiles, static_cast<cudaStream_t>(stream)));
  }
  CUDA_TRY(gemm_launch(p, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_kernel_attention(const void* q, int ldq, const void* k, const void* v, int ldkv, void* o,
                         int ldo, int batch, int n_q, int n_kv, int n_heads, int d_head, int impl,
                         void* stream) {
  return sgd_kernel_attention_hs(q, ldq, k, v, ldkv, d_head, o, ldo, batch, n_q, n_kv, n_heads, d_head,
                                 impl, stream);
}

int sgd_kernel_attention_hs(const void* q, int ldq, const void* k, const void* v, int ldkv, int head_stride,
                            void* o, int ldo, int batch, int n_q, int n_kv, int n_heads, int d_head,
                            int impl, void* stream) {
  if (impl < 0 || impl > 3) return fail(SGD_ERR_ARG, "attention: impl must be in 0..3");
  AttnPlan plan;
  plan.p = AttnParams{H16(q), ldq, H16(k), H16(v), ldkv, static_cast<f16*>(o), ldo,
                      batch, n_q, n_kv, n_heads, d_head, impl, head_stride};
  const char* why = "";
  const int rc = attn_plan(plan, &why);
  if (rc) return fail(rc == -1 ? SGD_ERR_ARG : (rc == -5 ? SGD_ERR_CUDA : SGD_ERR_SHAPE), why);
  CUDA_TRY(attn_launch(plan, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_kernel_norm(const float* h, void* out, int rows, int d, int kind, const void* g, const void* b,
                    const float* shift, const float* scale, int ld_mod, int rows_per_batch, float eps,
                    void* stream) {
  if (!h || !out || rows < 1 || d < 4 || d % 4 || d > 4096 || kind < 0 || kind > 2)
    return fail(SGD_ERR_ARG, "norm: bad arguments (d must be a multiple of 4, <= 4096)");
  if ((shift == nullptr) != (scale == nullptr) || (shift && rows_per_batch < 1))
    return fail(SGD_ERR_ARG, "norm: shift and scale go together, rows_per_batch >= 1");
  if (!al16(h) || (reinterpret_cast<uintptr_t>(out) & 7u))
    return fail(SGD_ERR_ARG, "norm: h must be 16-byte and out 8-byte aligned");
  NormParams p{h, static_cast<f16*>(out), rows, d, kind, B16(g), B16(b), shift, scale, ld_mod,
               rows_per_batch > 0 ? rows_per_batch : 1, eps};
  CUDA_TRY(norm_launch(p, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_kernel_frozen_run(float* h, const void* const* caches, int n_caches, int64_t n, void* stream) {
  if (!h || !caches || n_caches < 1 || n_caches > kMaxRun || n < 0 || n % 8 || !al16(h))
    return fail(SGD_ERR_ARG, "frozen_run: bad arguments");
  FrozenParams p{};
  p.h = h;
  p.n = n;
  p.n_caches = n_caches;
  for (int i = 0; i < n_caches; ++i) {
    if (!caches[i] || !al16(caches[i])) return fail(SGD_ERR_ARG, "frozen_run: null or misaligned cache");
    p.caches[i] = H16(caches[i]);
  }
  CUDA_TRY(frozen_launch(p, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_selftest_wait_timeout(void* stream) {
  int* p = device_status_ptr();
  if (!p) return fail(SGD_ERR_CUDA, "status word unavailable");
  CUDA_TRY(wait_selftest_launch(p, SGD_SELFTEST_TIMEOUT_CODE, static_cast<cudaStream_t>(stream)));
  return SGD_OK;
}

int sgd_kernel_gemm_stat_slots(int M, int N, int K, const sgd_epilogue_args* ea, int variant, int* slots) {
  if (!slots || !ea) return fail(SGD_ERR_ARG, "null argument");
  // the tile width is chosen on the host from the shape alone; plan with dummy aligned operands
  static const uint4 dummy[1] = {};
  sgd_epilogue_args e = *ea;
  GemmPlan p;
  p.encode = false;
  int rc = kernel_gemm_plan(dummy, K, dummy, K, M, N, K, &e, variant, p);
  if (rc) return rc;
  *slots = p.simt ? 0 : 2 * ((N + p.bn - 1) / p.bn);
  return SGD_OK;
}

int sgd_kernel_f16_clamped(int* clamped_host) {
  if (!clamped_host) return fail(SGD_ERR_ARG, "null argument");
  *clamped_host = 0;
  for (auto accessor : f16_clamp_flags()) {
    unsigned int* p = accessor();
    if (!p) return fail(SGD_ERR_CUDA, "fp16 clamp flag unavailable");
    unsigned int v = 0;
    CUDA_TRY(cudaMemcpy(&v, p, sizeof(v), cudaMemcpyDeviceToHost));
    if (v) {
      *clamped_host = 1;
      CUDA_TRY(cudaMemset(p, 0, sizeof(v)));
    }
  }
  return SGD_OK;
}

int sgd_kernel_status(int* status_host) {
  if (!status_host) return fail(SGD_ERR_ARG, "null argument");
  int* p = device_status_ptr();
  if (!p) return fail(SGD_ERR_CUDA, "status word unavailable");
  CUDA_TRY(cudaMemcpy(status_host, p, sizeof(int), cudaMemcpyDeviceToHost));
  if (*status_host) CUDA_TRY(cudaMemset(p, 0, sizeof(int)));
  return SGD_OK;
}

}  // extern "C"
