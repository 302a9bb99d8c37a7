/*
 * wam.h — C ABI of the GB300-native WAMachine hot path.
 *
 * The library runs the iterative flow denoising loop of a World Action Model: a DiT-style
 * transformer over the joint [observation ; future-video-latent ; action] token sequence,
 * integrated with explicit Euler steps, and the three state-adaptation mechanisms of
 * "Efficient World Action Model Inference with Adaptive Intermediate States"
 * (arXiv 2609.34608):
 *   - Trajectory Remapping (TR), §3.1, Eqs. 1-2 and App. B.1 Eq. 12,
 *   - Observation Rebinding (OR), §3.2, Eq. 4 and the kappa rule,
 *   - Residual Rescaling (RR), §3.3, Eqs. 5-9,
 * coordinated as described in §3.4.  The paper does not define the denoiser (it cites DiT);
 * the network implemented here is fixed by the weight layout documented below.
 *
 * Conventions for every call
 *   - Return value: WAM_OK or one WAM_ERR_* code.  No call aborts or throws across the ABI;
 *     wam_last_error() returns a message for the last failure on a context.
 *   - Buffers are owned by the caller.  Each buffer argument may be a host pointer or a device
 *     pointer of the current device; the library detects which (CUDA pointer attributes).
 *     Host buffers are copied in / out inside the call; a call with a host output returns
 *     only after the output has been written.  With device buffers only, a call returns
 *     once its work is enqueued on the context's stream.
 *   - Contexts and states own their device memory.  A context is used from one host thread
 *     at a time; it is not thread-safe.  Different contexts may be driven from different host
 *     threads at the same time (they share no mutable state).
 *   - All float buffers are IEEE float32, row-major, contiguous.
 *
 * Layouts (B = episodes in a state, No/Nv/Na = observation/video/action tokens,
 *          d = model width, T = Nv*video_dim + Na*action_dim)
 *   obs        [B, No, d]   already-encoded observation tokens (the condition c of §3.2)
 *   trajectory [B, T]       video values (token-major, video_dim each) then action values
 *   actions    [B, Na, action_dim]
 *   video      [B, Nv, video_dim]
 */
#ifndef WAM_H_
#define WAM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------------------- */
#define WAM_OK 0
#define WAM_ERR_INVALID_ARG 1  /* null / mis-sized / out-of-range argument */
#define WAM_ERR_BAD_STATE 2    /* call not valid for the state's current phase */
#define WAM_ERR_OOM 3          /* device allocation failed */
#define WAM_ERR_CUDA 4         /* a CUDA runtime call or kernel launch failed */
#define WAM_ERR_TIMEOUT 5      /* a bounded device-side wait gave up (kernel returned early) */
#define WAM_ERR_UNSUPPORTED 6  /* configuration outside what the kernels implement */

/* ---- precision ---------------------------------------------------------------------- */
#define WAM_PREC_FP32 0  /* SIMT float32 everywhere */
#define WAM_PREC_BF16 1  /* bf16 tensor-core GEMMs / attention, float32 residual stream */

/* ---- RR policies (App. B.1, paragraph after Table 5) -------------------------------- */
#define WAM_RR_OFF 0         /* every step runs all layers */
#define WAM_RR_ALL_PATHS 1   /* reuse allowed on every step once a layer state exists */
#define WAM_RR_PREFIX_PATH 2 /* reuse only on the anticipatory path after its first full step */

/* ---- adapt statuses (per episode, written by wam_adapt_state) ------------------------ */
#define WAM_ADAPT_TR_INIT 1           /* remapped init at b0; an anticipatory prefix may run */
#define WAM_ADAPT_TR_INIT_NO_PREFIX 2 /* remapped init; kappa reached kappa_max: skip the prefix */
#define WAM_ADAPT_COLD_INIT 3         /* fresh episode: noise at stage 0 */
#define WAM_ADAPT_REBIND_ACCEPT 4     /* consistency passed: real condition bound, state kept */
#define WAM_ADAPT_REBIND_RESTART 5    /* consistency failed: restart from the remapped init */
#define WAM_ADAPT_REFRESH 6           /* no prefix ran: real condition bound at b0, kappa = 0 */

/* entry_stage value that starts an episode afresh from noise (the first replan, §3.1) */
#define WAM_ENTRY_COLD (-1)

/*
 * Model + method profile.  Plain values, copied by wam_create.
 *
 * Schedule: sigma_k = s t_k / (1 + (s-1) t_k), t_k = 1 - k/K, k = 0..K (s = sched_shift;
 * s = 1 is linear flow time).  Step k integrates x_{k+1} = x_k + (sigma_{k+1}-sigma_k) v_k.
 *
 * TR (§3.1): the retained stage r (tr_retain_stage, -1 = same as the entry stage) and entry
 * stage b0 (tr_entry_stage, per-episode override in wam_adapt_state) with r >= b0 of the
 * replan that produced the state and r < K.  tr_normalize = 1 uses the unit-RMS normaliser of
 * Eq. 12, 0 the identity.  tr_video_mode = 0 remaps video without a temporal shift, 1 fills
 * video with fresh noise (the Motus profile of App. B.1).  Action slots shift by the executed
 * count; uncovered tail slots get fresh noise sigma_b0 * eps.
 *
 * RR (§3.3): boundaries 0 < rr_q < rr_s < rr_e < n_layers; factor clamp [alpha_min, alpha_max]
 * and epsilon of Eq. 7; gate thresholds of Eq. 8.  Branches (joint execution): observation and
 * video rows form one branch, action rows the other; each gets its own alpha and the middle
 * layers are skipped only if both pass.
 *
 * Independent execution (§3.3, App. B.1 Fast-WAM-IDM profile): n_video = 0 makes an
 * action-only model and n_action = 0 a video-only one (not both).  Such a model is one branch:
 * all of its rows share one alpha and one gate decision, its TR direction is normalised over
 * its own trajectory, and its context keeps its own replan state, schedule (sched_shift) and
 * retained / entry stages.  Two contexts then form the video and action branches; video_dim and
 * action_dim stay >= 1 and the unused branch's embedding / output weights stay in the weight
 * layout (ignored).  wam_continue_many advances both concurrently.
 *
 * OR (§3.2): Eq. 4 over or_n_components (1..4) equal contiguous blocks of observation tokens
 * with per-component scale or_deltas[m] and weight or_weights[m]; accept iff S < or_tau and
 * kappa < or_kappa_max.
 */
typedef struct wam_config {
  int32_t n_layers, d_model, n_heads, mlp_ratio;
  int32_t n_obs, n_video, video_dim, n_action, action_dim;
  int32_t n_steps;   /* K native solver steps */
  int32_t precision; /* WAM_PREC_* */
  int32_t batch_max; /* largest state batch this context will run */
  float sched_shift;
  int32_t tr_entry_stage, tr_retain_stage, tr_normalize, tr_video_mode;
  int32_t rr_policy, rr_q, rr_s, rr_e;
  float rr_alpha_min, rr_alpha_max, rr_eps, rr_gamma_cos, rr_gamma_fit;
  float or_tau;
  int32_t or_kappa_max, or_n_components;
  float or_deltas[4];
  float or_weights[4];
} wam_config;

/* Reuse statistics, App. D.2 Eqs. 14-15 (counts; rates are ratios of these). */
typedef struct wam_stats {
  int64_t n_attempt;     /* RR checks evaluated against a retained layer state */
  int64_t n_reuse;       /* accepted checks that skipped the middle layers */
  int64_t b_skip;        /* skipped layer evaluations */
  int64_t b_dense;       /* full-depth layer count of RR-enabled steps */
  int64_t n_start;       /* anticipatory prefixes started (rebinding attempts) */
  int64_t n_bind;        /* prefixes accepted and used */
  int64_t n_noninitial;  /* replans after the first (TR inits) */
  int64_t n_episode_steps;  /* denoising steps executed, summed over episodes */
  int64_t n_layer_evals;    /* transformer layer evaluations, summed over episodes */
  int64_t n_kernel_launches;/* kernels launched by this context */
} wam_stats;

/* One record per (episode, denoising step) of the latest wam_sample_cold / wam_continue. */
typedef struct wam_step_record {
  int32_t episode, stage;
  int32_t rr_active;  /* step ran on an RR-enabled path */
  int32_t rr_attempt; /* gate evaluated */
  int32_t rr_accept;  /* middle layers skipped */
  int32_t pad_;
  float alpha[2], cos[2], fit[2]; /* per branch: 0 = obs+video rows, 1 = action rows */
} wam_step_record;

typedef struct wam_ctx wam_ctx;
typedef struct wam_state wam_state;

/*
 * Number of floats in the flat weight buffer for cfg, or 0 if cfg is invalid.
 * Weight order (matrices [in, out], y = x W + b):
 *   obs_w[d,d] obs_b[d] vid_w[video_dim,d] vid_b[d] act_w[action_dim,d] act_b[d] pos[N,d]
 *   t_w1[256,d] t_b1[d] t_w2[d,d] t_b2[d]
 *   per layer: ada_w[d,6d] ada_b[6d] qkv_w[d,3d] qkv_b[3d] out_w[d,d] out_b[d]
 *              up_w[d,r d] up_b[r d] down_w[r d,d] down_b[d]          (r = mlp_ratio)
 *   final_ada_w[d,2d] final_ada_b[2d] vout_w[d,video_dim] vout_b[video_dim]
 *   aout_w[d,action_dim] aout_b[action_dim]
 * Network: tokens [obs W_o + b_o ; x_video W_v + b_v ; x_action W_a + b_a] + pos.
 * Conditioning c = SiLU(e W_t1 + b_t1) W_t2 + b_t2 with e = [cos(1000 sigma f), sin(1000 sigma f)],
 * f_j = 10000^(-j/128).  Layer modulations (shift1, scale1, gate1, shift2, scale2, gate2)
 * = SiLU(c) ada_w + ada_b; h += gate1 * Attn(LN(h)(1+scale1)+shift1) W_out;
 * h += gate2 * GELU_tanh(LN(h)(1+scale2)+shift2 W_up) W_down (biases included, LN eps 1e-6,
 * no affine; attention full, unmasked, scale 1/sqrt(d/heads)).  Output: LN(h)(1+scale)+shift
 * then vout on video rows, aout on action rows.
 */
size_t wam_weight_count(const wam_config* cfg);

/*
 * Create a context: validates cfg, uploads and converts the weights (host or device pointer,
 * n_weights == wam_weight_count(cfg)), allocates activation buffers for batch_max episodes.
 * stream: a cudaStream_t (NULL = legacy default stream).
 * Errors: INVALID_ARG (cfg or weights), UNSUPPORTED (shape the kernels cannot run), OOM, CUDA.
 */
int wam_create(const wam_config* cfg, const float* weights, size_t n_weights, void* stream,
               wam_ctx** out);
void wam_destroy(wam_ctx* ctx);
const char* wam_last_error(const wam_ctx* ctx);
int wam_set_stream(wam_ctx* ctx, void* stream);

/* Per-episode replan / denoising / layer state for `batch` episodes (1..batch_max).
 * A state belongs to its context: destroy every state before destroying the context. */
int wam_state_create(wam_ctx* ctx, int32_t batch, wam_state** out);
void wam_state_destroy(wam_state* st);

/*
 * First replan of every episode (§3.1: it starts from fresh noise): x_0 = noise [B,T] at stage 0
 * under obs [B,No,d], then n_steps (1..K) Euler steps.  Resets kappa and the RR layer state.
 * actions_out [B,Na,action_dim] (nullable) receives the latent's action part after the
 * last step (the denoised actions when n_steps == K).
 */
int wam_sample_cold(wam_ctx* ctx, wam_state* st, const float* obs, const float* noise,
                    int32_t n_steps, float* actions_out);

/*
 * Adapt the retained state to a new planning context, per episode:
 *   finished replan (stage K): Trajectory Remapping, Eqs. 1-2 — direction from x^r and x_bar,
 *       remapped init at b0 = entry_stage[b] (NULL: cfg.tr_entry_stage) with the action
 *       horizon shifted by executed_shift[b] (>= 0), fresh slots sigma_b0 * fresh_noise;
 *       new_obs becomes the bound condition (a prediction, for an anticipatory prefix, or the
 *       real observation).  Status TR_INIT, or TR_INIT_NO_PREFIX when kappa == kappa_max.
 *   replan in flight: Observation Rebinding, §3.2 — executed_shift[b] must be 0; if a prefix
 *       ran since the last binding, S (Eq. 4) compares the bound condition with new_obs;
 *       S < tau and kappa < kappa_max binds new_obs and keeps the denoising state
 *       (REBIND_ACCEPT, kappa+1), otherwise the episode restarts from its remapped init
 *       under new_obs (REBIND_RESTART, kappa = 0).  With no prefix steps: REFRESH.
 *   entry_stage[b] == WAM_ENTRY_COLD: fresh episode, x_0 = fresh_noise[b] at stage 0 (COLD_INIT).
 * new_obs [B,No,d]; executed_shift [B] (NULL = all 0); fresh_noise [B,T] standard normal
 * (required when any episode remaps or starts cold); status_out [B] (nullable).
 * Errors: INVALID_ARG, BAD_STATE (retained stage unavailable, shift on a rebind).
 */
int wam_adapt_state(wam_ctx* ctx, wam_state* st, const float* new_obs,
                    const int32_t* executed_shift, const int32_t* entry_stage,
                    const float* fresh_noise, int32_t* status_out);

/*
 * Advance each episode n_steps[b] (>= 0, stage + n <= K) Euler steps under its bound
 * condition, with Residual Rescaling per cfg.rr_policy.  Episodes that reach stage K become
 * finished replans (x_bar = x_K).  actions_out [B,Na,action_dim], video_out [B,Nv,video_dim]
 * (both nullable) receive every episode's current latent after the call.
 */
int wam_continue(wam_ctx* ctx, wam_state* st, const int32_t* n_steps, float* actions_out,
                 float* video_out);

/*
 * wam_continue on n (>= 1) distinct contexts at once, each from its own host thread (the
 * calling thread runs the first), so the branches of independent execution overlap on the GPU
 * when their contexts use different streams.  Element i of every array belongs to context i:
 * states[i] belongs to ctxs[i]; n_steps[i] has states[i]'s batch entries; actions_out and
 * video_out (each nullable, as are their elements) as in wam_continue.  Results are those of
 * n separate wam_continue calls.  status_out [n] (nullable) receives each call's status; the
 * return value is the first non-zero of them, or WAM_OK.  Each context's last error names its
 * own failure.  Errors: INVALID_ARG (null arrays, a state of another context, a context twice).
 */
int wam_continue_many(int32_t n, wam_ctx* const* ctxs, wam_state* const* states,
                      const int32_t* const* n_steps, float* const* actions_out,
                      float* const* video_out, int32_t* status_out);

/* Reuse statistics accumulated on the context since creation / the last reset. */
int wam_get_stats(wam_ctx* ctx, wam_stats* out);
int wam_reset_stats(wam_ctx* ctx);

/* Per-step records of the latest sampling call: copies min(capacity, available) records. */
int wam_state_log(const wam_state* st, wam_step_record* out, int32_t capacity, int32_t* n_out);

/* ---- state export / import (checkpoint + parity inspection) ------------------------- */
#define WAM_FIELD_X 0        /* current latent            [B,T]     */
#define WAM_FIELD_X_STAGE 1  /* latent at stage `index`   [B,T]     (index 0..K) */
#define WAM_FIELD_V_STEP 2   /* velocity of the step from stage `index` [B,T] (index 0..K-1) */
#define WAM_FIELD_X_INIT 3   /* remapped init x^{b0}      [B,T]     */
#define WAM_FIELD_OBS 4      /* bound condition           [B,No,d]  */
#define WAM_FIELD_RR_P 5     /* retained probe residual p_a  [B,N,d] */
#define WAM_FIELD_RR_R 6     /* retained middle residual R_a [B,N,d] */
/* Host-side per-episode scalars: 8 int32 per episode:
 * stage, hist_from, b0, kappa, finished, since_bind, path (0 cold 1 prefix 2 refresh), rr_valid */
#define WAM_FIELD_META 7
int wam_state_read(wam_ctx* ctx, const wam_state* st, int32_t field, int32_t index, void* out,
                   size_t n_bytes);
int wam_state_write(wam_ctx* ctx, wam_state* st, int32_t field, int32_t index, const void* in,
                    size_t n_bytes);

/* Wait for the context's stream; returns a pending device-side error (e.g. TIMEOUT). */
int wam_sync(wam_ctx* ctx);

/* Kernel-class timing spans recorded with CUDA events on the context's stream. */
#define WAM_KCLASS_GEMM 0      /* tcgen05 / SIMT projections */
#define WAM_KCLASS_ATTN 1      /* attention */
#define WAM_KCLASS_NORM 2      /* LN-modulate */
#define WAM_KCLASS_COND 3      /* conditioning GEMVs */
#define WAM_KCLASS_ADAPT 4     /* TR remap / OR score / bind (wam_adapt_state) */
#define WAM_KCLASS_EMBED 5     /* token embedding, observation cast */
#define WAM_KCLASS_FINAL 6     /* final layer + Euler update */
#define WAM_KCLASS_RR_PROBE 7  /* RR probe reductions and gate */
#define WAM_KCLASS_RR_APPLY 8  /* RR gather, injection / refresh */
#define WAM_KCLASS_COUNT 9
typedef struct wam_kclass_timing {
  int64_t launches;
  double ms;          /* summed event-measured duration */
  double flops;       /* algorithmic flops of those launches */
  double bytes;       /* algorithmic bytes of those launches */
} wam_kclass_timing;
/* enable != 0 starts recording (clears previous spans); reading synchronizes the stream. */
int wam_profile_enable(wam_ctx* ctx, int32_t enable);

/*
 * One task of a fused row-chain launch (wam_set_layer_fusion), recorded while profiling is on:
 * kind 0 out-projection, 1 LN before the MLP, 2 MLP up, 3 MLP down, 4 LN of the next block, 5 QKV
 * projection; m = 128-row block, j = column tile (or 32-row quarter for LN); times are the GPU's
 * global timer in ns: task taken, dependency satisfied (operands requested), epilogue start,
 * completion published.
 */
typedef struct {
  int32_t launch, cta, kind, m, j, pad;
  uint64_t t_take, t_dep, t_epi0, t_epi1;
} wam_chain_task;

/*
 * Copies up to `capacity` recorded chain tasks (in launch order) since profiling was enabled into
 * out (host memory) and their count into *n_out.  Synchronises the context's stream.
 * WAM_ERR_INVALID_ARG for null pointers.
 */
int wam_profile_chain_trace(wam_ctx* ctx, wam_chain_task* out, int32_t capacity, int32_t* n_out);
int wam_profile_read(wam_ctx* ctx, wam_kclass_timing* out /* [WAM_KCLASS_COUNT] */);

/*
 * State-continuity diagnostics (paper App. E), computed on the device in float64.  Inputs may be
 * host or device pointers; the calls synchronise the context's stream and return the values.
 *
 * wam_diag_similarity: cosine similarity <a,b>/(|a||b|) and relative L2 distance |a-b|/|b| of
 *   two vectors of n floats (App. E: the latent x_t^r of the current replan against the
 *   preceding replan's x_{t-1}^r at the same stage r, the preceding one being b).  A zero-norm
 *   input gives cos 0; |b| = 0 gives rel_l2 0 if a == b, else HUGE_VAL.
 * wam_diag_action_rmse: sqrt(mean over rows j and the first `dims` of each row's `row_len`
 *   values of (a - b)^2) (App. E Eq. 17 with dims = 6; actions [n_rows, row_len]).
 * wam_diag_layer_deltas: for one episode of a state at its pending stage k (0 <= k < K), runs
 *   the full forward at sigma_k on its current latent and bound observation and writes
 *   out[l] = |h_{l+1} - h_l| / |h_l| for every layer l (h_0 = the token embedding), the hidden
 *   state change of App. E.  The state is not modified (context scratch only).
 * wam_diag_reuse_error: for one episode at its pending stage k with a retained RR layer state,
 *   the residual-reuse output error of App. E, E_out = |y_reuse - y_full| / |y_full| on identical
 *   inputs: y_full the full forward at sigma_k, y_reuse the forward whose middle layers [s, e) are
 *   replaced by h_s + alpha R_a (Eq. 9) with alpha per branch from Eq. 7 against the retained
 *   layer state, whatever the Eq. 8 checks say.  alpha_out [2] (nullable) receives the factors
 *   (0 for a branch the model does not have).  The state is not modified.  Errors:
 *   WAM_ERR_INVALID_ARG also when the profile has no RR boundaries; WAM_ERR_BAD_STATE also when
 *   the episode has no retained layer state yet.
 * n (resp. n_rows * row_len) is at most batch_max * tokens * d_model.  Errors:
 * WAM_ERR_INVALID_ARG (null, sizes), WAM_ERR_BAD_STATE (episode finished or not started).
 */
int wam_diag_similarity(wam_ctx* ctx, const float* a, const float* b, int64_t n, double* cos_out,
                        double* rel_l2_out);
int wam_diag_action_rmse(wam_ctx* ctx, const float* a, const float* b, int32_t n_rows,
                         int32_t row_len, int32_t dims, double* out);
int wam_diag_reuse_error(wam_ctx* ctx, wam_state* state, int32_t episode, double* e_out,
                         double* alpha_out);
int wam_diag_layer_deltas(wam_ctx* ctx, wam_state* state, int32_t episode,
                          double* out /* [n_layers] */);

/*
 * CUDA-graph replay of the layer stack (default on).  Each contiguous range of DiT layers a step
 * runs (all layers; or the head, the gathered middle and the tail around Residual Rescaling) is
 * captured into a CUDA graph the second time the same range, batch width and buffers occur, and
 * replayed from then on; host decisions (RR gate, OR rule, TR bookkeeping) stay outside the graphs,
 * as in the paper (§4, App. D).  enable = 0 launches every kernel individually (the ablation).
 * Results are identical either way.
 */
int wam_set_graph_replay(wam_ctx* ctx, int32_t enable);

/*
 * Device-side Residual Rescaling branching (default on).  When a denoising step has a single work
 * item whose RR check is attempted and the layer stack is replayed from graphs, the whole step
 * around the gate (layers before the probe end, the probe sums and the Eq. 8 check, the middle
 * layers under a graph conditional node that runs them only when the check fails, the injection
 * or refresh, and the tail layers) is one CUDA graph captured on its second use: the decision is
 * taken on the device and the host does not wait for it.  The decisions reach the step log and
 * the reuse statistics through a small ring copied after each call; wam_state_log and
 * wam_get_stats wait for the copies.  enable = 0 keeps the decision on the host (a read-back per
 * step).  Results are identical either way.  WAM_ERR_INVALID_ARG for a null context.
 */
int wam_set_device_branching(wam_ctx* ctx, int32_t enable);

/*
 * Fused row-chain launches (default off).  Between two attentions the work of the DiT blocks is
 * row-local: out-projection + gated residual, LN + modulation, MLP, gated residual, then the next
 * block's LN + modulation and QKV projection.  With enable != 0, bf16 models with the tensor-core
 * attention and a layer range of at most 16384 rows (episodes x tokens) run these as one
 * persistent tensor-core launch per block instead of six, with per-row-block dependencies.  The
 * arithmetic is the same either way (identical results).  Measured on one episode of the 12-block
 * d768 model the fused launch is slower than the separate ones, so it is off by default.
 * Returns WAM_ERR_INVALID_ARG for a null context.
 */
int wam_set_layer_fusion(wam_ctx* ctx, int32_t enable);

/*
 * Output tile width (64, 128 or 256 columns) the context's bf16 path uses for the GEMM
 * [M, K] x [K, N] with the given epilogue (WAM_EPI_*, or 4 for the QKV projection that also
 * writes V^T), chosen from the shape alone: 64 (residual projections, WAM_EPI_RESID_F32) while
 * 128-wide tiles cannot fill the SMs, 256 from
 * four waves of 256-wide tiles on, else 128.  When K % 128 == 0, 256-wide tiles, and 128-wide
 * tiles that fill four waves, run on CTA pairs sharing one two-SM MMA.  Every width and pairing
 * sums K in the same order, so the choice affects speed only.  Returns WAM_ERR_INVALID_ARG for a
 * null context,
 * WAM_ERR_UNSUPPORTED for the fp32 path.
 */
int wam_gemm_tile_width(const wam_ctx* ctx, int32_t M, int32_t N, int32_t K, int32_t epilogue);

#ifdef __cplusplus
}
#endif
#endif /* WAM_H_ */
