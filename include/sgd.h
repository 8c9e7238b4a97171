/*
 * sgd.h — C ABI of libsgd: one denoiser evaluation per diffusion step under a
 * static spectral layer-step schedule, on one NVIDIA GB300 (sm_103a).
 *
 * Method (paper: "Spectral-Guided Diffusion: Accelerating Inference via Static
 * Spectral Layer Scheduling"):
 *   - Sec. 3.1: a residual unit maps h_{l-1,s} to h_{l,s} = h_{l-1,s} + F_l(h_{l-1,s}; c_s).
 *     A unit with lifetime S_l is evaluated for s <= S_l; afterwards the stored
 *     update Delta_{l, r_l(s)} is added to the *current* residual stream.
 *   - Sec. 4.1, Eq. schedule: lifetimes come from weight-only scores (computed by the
 *     host; this library takes them as integers).
 *   - Sec. 4.2 and Algorithm 2: the dependency-closed active/frozen pattern of each
 *     step is replayed as one captured CUDA graph; active units compute their update,
 *     store it and add it; frozen units only add the stored update.
 *
 * Conventions for every entry point:
 *   - Pointers named *_dev are device pointers on the device that was current at
 *     sgd_create; *_host pointers are host pointers.  The caller owns every buffer
 *     it passes; the library owns caches, workspaces and graphs.
 *   - Every function returns an sgd_status (0 = success, negative = error) and never
 *     aborts or throws.  On error, sgd_last_error() describes it.
 *   - A context is not thread-safe: calls on one context must be serialised.
 *   - All weights are passed as bf16, row-major [out, in] for linear maps.  At
 *     sgd_create the projection weights are converted once into library-owned fp16
 *     copies scaled by a power of two (exact for every entry in fp16's normal range);
 *     the tensor cores then multiply fp16 operands with fp32 accumulation (same
 *     tcgen05 kind::f16 rate as bf16, 8x finer operand rounding).  Activations
 *     between kernels are fp16, the residual stream h and all reductions fp32.
 */
#ifndef SGD_H
#define SGD_H

#include <stddef.h>
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

typedef enum {
  SGD_OK = 0,
  SGD_ERR_ARG = -1,            /* null pointer, bad enum, bad alignment            */
  SGD_ERR_SHAPE = -2,          /* unsupported or inconsistent model shape          */
  SGD_ERR_SCHEDULE = -3,       /* lifetime outside [1,T] or an atomic group split  */
  SGD_ERR_CACHE_INVALID = -4,  /* step s called without steps 1..s-1 since reset   */
  SGD_ERR_CUDA = -5,           /* a CUDA runtime call failed                       */
  SGD_ERR_DEVICE_TIMEOUT = -6, /* a kernel's bounded wait expired (device status)  */
  SGD_ERR_OOM = -7,            /* device allocation failed                         */
  SGD_ERR_STATE = -8,          /* call order violated (e.g. step before schedule)  */
  SGD_ERR_RANGE = -9           /* an fp16 value was clamped to +-65504 (or NaN)    */
} sgd_status;

/* Input stage of the denoiser. */
typedef enum {
  SGD_STEM_TIME_ADD = 0,     /* h0 = z + sinusoid(t, d) on every token; z fp32 [B,N,d]   */
  SGD_STEM_PATCH = 1,        /* h0 = z W_stem^T + pos_emb; z fp32 [B,N,d_in]             */
  SGD_STEM_PATCH_TOKENS = 2, /* U-ViT: [sinusoid(t); class_emb[y]; z W_stem^T] + pos_emb */
  SGD_STEM_IDENTITY = 3,     /* h0 = z; z fp32 [B,N,d]                                   */
  SGD_STEM_EMBED = 4         /* h0 = embed[ids]; ids int32 [B,N]                         */
} sgd_stem_kind;

/* Residual block family; the branches of one block are units in graph order. */
typedef enum {
  SGD_BLOCK_PRENORM = 0,  /* {self-attention, MLP}, pre-norm                      */
  SGD_BLOCK_ADALN = 1,    /* {self-attention, MLP}, AdaLN-Zero modulation + gates */
  SGD_BLOCK_XATTN = 2     /* {self-attention, cross-attention, MLP}, pre-norm     */
} sgd_block_kind;

typedef enum {
  SGD_NORM_RMS = 0,       /* x * rsqrt(mean(x^2) + eps) * g                */
  SGD_NORM_LN = 1,        /* (x - mu) * rsqrt(var + eps) * g + b           */
  SGD_NORM_LN_PLAIN = 2   /* LayerNorm without affine (AdaLN blocks)       */
} sgd_norm_kind;

typedef enum {
  SGD_MLP_SWIGLU = 0,     /* W_2 (silu(W_1[:f] x) * W_1[f:] x)   */
  SGD_MLP_GELU_TANH = 1,  /* W_2 gelu_tanh(W_1 x)                */
  SGD_MLP_GELU_ERF = 2,   /* W_2 gelu_erf(W_1 x)                 */
  SGD_MLP_GEGLU = 3       /* W_2 (W_1[:f] x * gelu_erf(W_1[f:] x)) */
} sgd_mlp_kind;

typedef enum {
  SGD_HEAD_LINEAR = 0,       /* norm_f then W_head; fp32 out [B, N - n_prefix, out_channels] */
  SGD_HEAD_ADALN_LINEAR = 1, /* AdaLN(final) then W_head; fp32 out, first out_channels      */
  SGD_HEAD_IDENTITY = 2,     /* out = h_L; fp32 [B, N, d]                                  */
  SGD_HEAD_LOGITS = 3        /* RMSNorm then W_head; fp16 logits [B, N, d_out]            */
} sgd_head_kind;

/* Debug flag: run every GEMM on the plain SIMT kernel instead of tcgen05. */
#define SGD_FLAG_SIMT_GEMM 1
/* Run every attention on the mma.sync kernel instead of tcgen05 (d_head 64 / 128). */
#define SGD_FLAG_MMA_SYNC_ATTENTION 2
/* (Flag bit 4 is not defined; sgd_create rejects it.) */
/* Use 64-element K-blocks (4 stages, 128-byte swizzle) in the tcgen05 GEMMs. */
#define SGD_FLAG_GEMM_BK64 8
/* Launch a step's kernels with programmatic dependent launch: each kernel's launch and
 * prologue overlap the previous kernel's tail (by default a kernel starts only after the
 * previous one has finished).  Measured on GB300 it gains nothing on the mid-size models
 * and loses 1.5% on the LLaDA-8B-shaped step, whose clock falls under the power cap. */
#define SGD_FLAG_PDL 16
/* Fold RMSNorm / LayerNorm pre-norms into the GEMMs that follow them (Algorithm 2's
 * Norm -> projection as one tcgen05 GEMM: the gain folded into the weight, the row
 * statistics applied in the epilogue, emitted by the previous writer of the residual stream
 * with an fp16 copy of it) instead of running a norm kernel first.  Off by default: measured
 * on GB300 it is slower (LLaDA-8B-shaped step -2% under the power cap, U-ViT / SDXL-shaped
 * -7 to -8%); results agree with the default path within fp16 rounding. */
#define SGD_FLAG_FOLD_NORM 32

typedef struct {
  int stem, block, norm, mlp, head;   /* enums above                                   */
  int n_blocks;                       /* residual blocks (<= 64)                       */
  int d, n_heads, d_head, d_ff;       /* width, heads, head dim (64, 72, 128), MLP f   */
  int batch, n_tokens;                /* B, N (tokens per sample inside the blocks)    */
  int n_prefix;                       /* U-ViT time/class tokens ahead of the patches  */
  int d_in;                           /* channels of the input state                   */
  int d_out;                          /* rows of W_head                                */
  int out_channels;                   /* channels written per output token             */
  int n_skips;                        /* U-ViT long skips (n_blocks = 2 n_skips + 1)    */
  int ctx_len, d_ctx;                 /* cross-attention context (SDXL)                 */
  int vocab, n_classes, t_freq;       /* token / class tables, DiT timestep frequencies */
  int rope;                           /* 1: rotate-half RoPE on q and k                 */
  float rope_theta, eps;
  int flags;                          /* SGD_FLAG_*                                     */
} sgd_model_desc;

/* Per-block weights (device, bf16, every pointer 16-byte aligned, else sgd_create returns
 * SGD_ERR_ARG).  Unused entries may be NULL. */
typedef struct {
  const void* norm1_w; const void* norm1_b;   /* [d]                                  */
  const void* w_qkv;                          /* [3d, d]: rows Q, then K, then V      */
  const void* w_o;                            /* [d, d]                               */
  const void* normx_w; const void* normx_b;   /* [d] cross-attention LayerNorm        */
  const void* wx_q;                           /* [d, d]                               */
  const void* wx_kv;                          /* [2d, d_ctx]: rows K, then V          */
  const void* wx_o;                           /* [d, d]                               */
  const void* norm2_w; const void* norm2_b;   /* [d]                                  */
  const void* w_1;                            /* [2f, d] gated (first f rows = gate/a) or [f, d] */
  const void* w_2;                            /* [d, f]                               */
  const void* w_mod;                          /* [6d, d] AdaLN: shift1 scale1 gate1 shift2 scale2 gate2 */
} sgd_block_weights;

/* Model weights (device, bf16, 16-byte aligned like the per-block ones). */
typedef struct {
  const sgd_block_weights* blocks;  /* host array of n_blocks entries (copied)     */
  const void* w_stem;               /* [d, d_in]                                   */
  const void* pos_emb;              /* [N, d]                                      */
  const void* w_t1; const void* w_t2; /* DiT timestep MLP: [d, t_freq], [d, d]    */
  const void* class_emb;            /* [n_classes, d]                              */
  const void* const* skip_w;        /* host array of n_skips device pointers [d, 2d] */
  const void* normf_w; const void* normf_b; /* [d]                                 */
  const void* w_modf;               /* [2d, d] DiT final AdaLN: shift, scale       */
  const void* w_head;               /* [d_out, d]                                  */
  const void* embed;                /* [vocab, d]                                  */
} sgd_weights;

/* Per-step conditioning (device pointers; NULL when the model has none). */
typedef struct {
  const int32_t* class_ids;  /* [B]                   */
  const void* ctx;           /* bf16 [B, ctx_len, d_ctx] */
} sgd_cond;

typedef struct {
  int n_units;          /* residual branches (units) in graph order            */
  int n_patterns;       /* distinct active sets of the current schedule          */
  int n_graphs;         /* captured graphs (patterns x cache-refresh variants)   */
  int T;                /* horizon of the current schedule (0 if none)            */
  int64_t layer_steps;  /* sum over steps of active units                         */
  size_t cache_bytes;   /* device bytes of the per-unit update caches (fp16)      */
  size_t workspace_bytes;
  size_t weight_bytes;  /* device bytes of the library's fp16 projection weights  */
  int policy;           /* SGD_POLICY_STATIC or SGD_POLICY_DRIFT                  */
  int n_groups;         /* scheduled (atomic) groups of the current schedule      */
  int64_t graph_steps;  /* drift policy: steps replayed from the graph library    */
  int64_t eager_steps;  /* drift policy: steps run op by op (pattern not in it)   */
} sgd_info;

typedef struct sgd_ctx sgd_ctx;

/*
 * sgd_create — validate the model shape, borrow the weights, make the fp16 projection
 * copies, allocate caches and workspaces on the current device.  The model is the
 * pretrained network of the problem statement (Sec. 3.1: a stack of residual units
 * h_{l,s} = h_{l-1,s} + F_l(h_{l-1,s}; c_s) evaluated once per sampler step); the context
 * holds what the executor of Sec. 4.2 keeps across steps (per-unit update caches,
 * captured graphs).
 * desc, w: host structs (copied).  Weight pointers: device, 16-byte aligned; norm
 * gains, embeddings, stem, conditioning and small-head weights are read in place and
 * must stay valid and unchanged for the context's lifetime.
 * Errors: SGD_ERR_ARG (null/misaligned), SGD_ERR_SHAPE, SGD_ERR_OOM, SGD_ERR_CUDA.
 */
SGD_API int sgd_create(const sgd_model_desc* desc, const sgd_weights* w, sgd_ctx** out);

/*
 * sgd_set_schedule — install per-unit lifetimes (Sec. 4.1, Eq. schedule) with their
 * atomic dependency groups (Sec. 3.1: dependency-coupled operations form atomic,
 * dependency-closed units).  Compiles the per-step active lists, captures one graph
 * per distinct active pattern (plus a variant for the step at which a pattern's
 * units store their final update), and resets the trajectory.
 * lifetimes_host: int32 [n_units], each in [1, T].  group_of_unit_host: int32
 * [n_units] group ids; all members of a group must share one lifetime.
 * Units are the residual branches in graph order: per block attn[, xattn], mlp.
 * Errors: SGD_ERR_SCHEDULE (bad lifetime, split group, n_units mismatch), SGD_ERR_CUDA.
 */
SGD_API int sgd_set_schedule(sgd_ctx* ctx, int T, int n_units, const int32_t* lifetimes_host,
                     const int32_t* group_of_unit_host);

/*
 * sgd_step — one denoiser evaluation at step `step` (Algorithm 2), asynchronous on
 * `stream` (a cudaStream_t).  step must be 1 (starts a trajectory) or last_step + 1.
 * state_in_dev: fp32 [B, N_in, d_in], or int32 ids [B, N] for SGD_STEM_EMBED.
 * out_dev: fp32 [B, N_out, out_channels] or fp16 logits [B, N, d_out].
 * timestep: t_s fed to the stem / conditioning.  cond: see sgd_cond (may be NULL).
 * Errors: SGD_ERR_STATE (no schedule), SGD_ERR_CACHE_INVALID (out-of-order step),
 * SGD_ERR_ARG, SGD_ERR_CUDA.  Kernel timeouts surface through sgd_check_device.
 */
SGD_API int sgd_step(sgd_ctx* ctx, const void* state_in_dev, void* out_dev, float timestep,
             const sgd_cond* cond, int step, void* stream);

/*
 * sgd_step_host — sgd_step with host buffers: copies the state (and conditioning
 * given as host pointers) to device, runs the step and copies the output back, all
 * on `stream`; returns after the output has arrived in out_host.  Pinned host
 * buffers give asynchronous copies.
 */
SGD_API int sgd_step_host(sgd_ctx* ctx, const void* state_in_host, void* out_host, float timestep,
                  const int32_t* class_ids_host, const void* ctx_host, int step, void* stream);

/*
 * sgd_step_host_async — sgd_step_host without the final wait: the input copy and the
 * step are queued on `stream`.  A pinned out_host (page-locked memory the runtime maps into
 * the device's address space, e.g. from cudaHostAlloc / cudaMallocHost) is written by the
 * step's output kernel directly, over the host link; any other out_host gets a copy on a
 * library-owned copy stream from a double-buffered device output, overlapping the compute
 * of step s + 1.  in_host should be pinned and must stay unchanged until the step's input
 * copy has run; out_host must not be read until sgd_host_wait returns.  Writes and copies
 * land in call order, so a later step may name the same out_host.
 */
SGD_API int sgd_step_host_async(sgd_ctx* ctx, const void* state_in_host, void* out_host,
                                float timestep, const int32_t* class_ids_host, const void* ctx_host,
                                int step, void* stream);

/* sgd_host_wait — wait until every output queued by sgd_step_host_async is in host memory. */
SGD_API int sgd_host_wait(sgd_ctx* ctx);

/* sgd_get_active_mask — the active set A_s of Sec. 3.1 / Algorithm 2 (unit u is evaluated
 * at step s iff s <= S_u): mask_host[u] = 1 iff unit u is evaluated at `step` (1..T).
 * Under the drift policy (App. B.1): the mask step `step` ran with (steps run since the
 * last reset).  mask_host: uint8 [n_units], n_units must equal the model's.
 * Errors: SGD_ERR_ARG, SGD_ERR_STATE (no schedule or step not yet run under drift). */
SGD_API int sgd_get_active_mask(const sgd_ctx* ctx, int step, uint8_t* mask_host, int n_units);

/* sgd_get_info — sizes and schedule statistics. */
SGD_API int sgd_get_info(const sgd_ctx* ctx, sgd_info* info);

/*
 * Execution modes (the execution ablation of Table tab:kernel):
 *   SGD_EXEC_JAGGED_GRAPH  default: one captured graph per active pattern, frozen units
 *                          launch no branch work (Sec. 4.2).
 *   SGD_EXEC_EAGER         the same per-step op list launched op by op from the host
 *                          (host-side skipping of frozen units, no graphs); with a 100%
 *                          schedule it is eager full inference.
 *   SGD_EXEC_PADDED_GRAPH  one graph per pattern that still evaluates every frozen
 *                          branch and discards its update (into a scratch residual),
 *                          then adds the cached update: all layer-steps executed.
 * All modes give bit-identical outputs.  Changing the mode resets the trajectory.
 */
enum { SGD_EXEC_JAGGED_GRAPH = 0, SGD_EXEC_EAGER = 1, SGD_EXEC_PADDED_GRAPH = 2 };
SGD_API int sgd_set_exec_mode(sgd_ctx* ctx, int mode);

/*
 * Active-set policies:
 *   SGD_POLICY_STATIC  default: unit u is active at step s iff s <= S_u (Algorithm 2).
 *   SGD_POLICY_DRIFT   the causal activation-drift baseline of App. B.1: after step s-1
 *                      the library has the lagged drift of every scheduled group's input,
 *                      d_g = ||h_{s-1} - h_{s-2}||_2 / (||h_{s-1}||_2 + 1e-8) (the residual
 *                      stream entering the group's first branch, over the whole batch),
 *                      and step s runs the m_s groups with the largest drift, m_s being the
 *                      static schedule's active count at s (ties to the lower group
 *                      index, groups numbered by their first unit).  Step 1 is full; at
 *                      step 2 no lagged drift exists yet and the m_2 lowest-indexed groups
 *                      run.  A frozen unit adds the update of its last active step, so
 *                      every active unit stores its update.  Each step s >= 3 waits on the
 *                      host for step s-1's drift sums (the routing is on the host, as in
 *                      the paper); a step whose active set is one of the static schedule's
 *                      patterns replays that pattern's graph, any other runs op by op.
 *                      Needs SGD_EXEC_JAGGED_GRAPH or SGD_EXEC_EAGER.
 * Changing the policy resets the trajectory.
 */
enum { SGD_POLICY_STATIC = 0, SGD_POLICY_DRIFT = 1 };
SGD_API int sgd_set_policy(sgd_ctx* ctx, int policy);

/*
 * sgd_get_drift — the lagged drifts the drift policy ranked to choose step `step`'s
 * active set, drift_host[g] for the n_groups groups (0 at steps 1 and 2).  Valid for
 * steps run since the last reset; SGD_ERR_STATE otherwise or under the static policy.
 */
SGD_API int sgd_get_drift(const sgd_ctx* ctx, int step, double* drift_host, int n_groups);

/* sgd_reset — start a new trajectory (Algorithm 2 starts at s = 1 with no stored updates):
 * the next step must be 1, and every cache counts as unwritten until its unit runs. */
SGD_API int sgd_reset(sgd_ctx* ctx);

/* sgd_check_device — synchronise `stream` and report a device-side status word set by
 * a kernel whose bounded wait expired (SGD_ERR_DEVICE_TIMEOUT), else the fp16 clamp flag
 * (SGD_ERR_RANGE: some fp16 activation, attention output or cached update left fp16's
 * finite range, or was NaN, and was stored clamped to +-65504 since the last check, so the
 * results are not to be trusted); clears what it reports. */
SGD_API int sgd_check_device(sgd_ctx* ctx, void* stream);

/* sgd_destroy — free everything the context owns (graphs, caches, workspaces; the state
 * the executor of Sec. 4.2 keeps across steps).  The borrowed weights are not touched. */
SGD_API void sgd_destroy(sgd_ctx* ctx);

/* sgd_last_error — message of the last failing call on this thread ("" if none).  ABI
 * plumbing with no counterpart in the paper: errors cross the boundary as status codes. */
SGD_API const char* sgd_last_error(void);

/*
 * sgd_compile_schedule — host-only schedule compiler (no device needed): validates
 * lifetimes/groups like sgd_set_schedule and returns, for steps s = 1..T,
 * pattern_of_step_host[s-1] (pattern id, numbered in order of first appearance),
 * writes_at_step_host[s-1] (number of units whose lifetime ends at s < T and which
 * therefore store their update at s), and *n_patterns.  Arrays are [T]; any of them
 * may be NULL.
 */
SGD_API int sgd_compile_schedule(int T, int n_units, const int32_t* lifetimes_host,
                         const int32_t* group_of_unit_host, int32_t* pattern_of_step_host,
                         int32_t* writes_at_step_host, int32_t* n_patterns);

/* Timing of one op of a profiled step. */
typedef struct {
  char name[48];        /* op label, e.g. "b3.attn.qkv_gemm"                */
  int kernel;           /* SGD_KERNEL_* id                                  */
  float ms;             /* CUDA-event duration on the launching stream      */
  double flops;         /* algorithmic FLOPs of the op                      */
  double bytes;         /* algorithmic DRAM bytes of the op                 */
} sgd_op_record;

enum {
  SGD_KERNEL_GEMM_TC = 0, SGD_KERNEL_GEMM_SIMT = 1, SGD_KERNEL_ATTENTION = 2,
  SGD_KERNEL_NORM = 3, SGD_KERNEL_FROZEN_RUN = 4, SGD_KERNEL_SMALL = 5, SGD_KERNEL_COUNT = 6
};

/*
 * sgd_step_profile — the same step as sgd_step, launched op by op outside the graph
 * with a CUDA event pair around every op on `stream`; synchronises and fills up to
 * max_records entries.  Same ordering rules as sgd_step.
 */
SGD_API int sgd_step_profile(sgd_ctx* ctx, const void* state_in_dev, void* out_dev, float timestep,
                     const sgd_cond* cond, int step, void* stream, sgd_op_record* records_host,
                     int max_records, int* n_records);

/*
 * sgd_sampler_update — z <- alpha z - beta eps, elementwise on n fp32 values (the
 * deterministic update of Sec. 3.1), asynchronous on `stream`.
 */
SGD_API int sgd_sampler_update(float* z_dev, const float* eps_dev, float alpha, float beta, int64_t n,
                       void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SGD_H */
