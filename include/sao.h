/*
 * sao.h -- C ABI of the SAO per-token RL loss head on one GB300 (sm_103a).
 *
 * The operations follow "Single-Rollout Asynchronous Optimization for Agentic
 * Reinforcement Learning" (arxiv 2607.07508):
 *   - sao_token_logprobs_fwd/bwd : log pi_theta(a_t|s_t) of Eq. 1-2 from the
 *     LM head (logits H W^T, log-softmax, gather), vocabulary-chunked so the
 *     [N, V] logits are never stored, and its gradient;
 *   - sao_policy_loss_fwd/bwd    : the DIS ratio of Eq. 2 against the rollout
 *     log-probs, the strict double-sided calibration f of Eq. 3 and the token
 *     objective of Eq. 1 (§3.1), with the clip-ratio counts of §4.4;
 *   - sao_advantages             : token-level GAE (Preliminaries) with the
 *     skip-observation link of Eq. 4-5 (§3.2) and the length-adaptive lambda
 *     of §4.1, as a reverse scan over packed trajectories;
 *   - sao_value_loss             : the value error (V - R)^2 (Preliminaries)
 *     and the explained-variance sums of §4.4.
 *
 * Conventions shared by every entry point:
 *   - Every array argument is a DEVICE pointer owned by the caller; the
 *     library never allocates, frees or keeps a pointer past the call.
 *   - Scratch space comes from the caller's workspace `ws` of `ws_bytes`
 *     bytes, 256-byte aligned, of at least sao_workspace_bytes(...) bytes.
 *     Its contents on entry do not matter; one workspace must not be used by
 *     two calls that overlap on the GPU.
 *   - Each call only enqueues kernels on `stream` (a cudaStream_t; NULL is
 *     the legacy default stream) and returns without waiting, unless checked
 *     mode is on (sao_set_checked), in which case it synchronises the stream
 *     and reports device-side validation failures as SAO_ERR_DEVICE_CHECK.
 *   - Errors are returned as sao_status; no exception crosses the ABI; the
 *     last error message is available from sao_last_error_string().
 *   - N is the number of packed tokens; row t of H predicts token y[t] (the
 *     caller does the shift). Per-token floating point arrays are fp32;
 *     token ids and cu_seqlens are int32; counts are int64.
 *   - Arrays are contiguous (row-major for matrices). Vectorised paths need
 *     16-byte aligned pointers; other alignments take a scalar path.
 */
#ifndef SAO_H_
#define SAO_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SAO_API __attribute__((visibility("default")))
#else
#define SAO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *sao_stream_t; /* a cudaStream_t */

typedef enum sao_status {
  SAO_OK = 0,
  SAO_ERR_INVALID_ARG = 1,  /* null pointer, bad scalar, misaligned workspace */
  SAO_ERR_SHAPE = 2,        /* inconsistent or unsupported sizes */
  SAO_ERR_WORKSPACE = 3,    /* ws_bytes smaller than required */
  SAO_ERR_UNSUPPORTED = 4,  /* dtype, or a device that is not sm_103 */
  SAO_ERR_CUDA = 5,         /* a CUDA runtime or driver call failed */
  SAO_ERR_DEVICE_CHECK = 6  /* checked mode: the device flagged bad input */
} sao_status;

typedef enum sao_dtype {
  SAO_F32 = 0,   /* fp32 H, W, dH (fp32 FMA path) */
  SAO_BF16 = 1   /* bf16 H, W, dH (tcgen05 tensor-core path, fp32 accumulate) */
} sao_dtype;

/* Per-token flag values written by sao_policy_loss_fwd (Eq. 3). */
#define SAO_FLAG_IN 0        /* 1 - eps_low < r < 1 + eps_high: kept, f(r) = r */
#define SAO_FLAG_LOW 1       /* r <= 1 - eps_low: masked, f(r) = 0 */
#define SAO_FLAG_HIGH 2      /* r >= 1 + eps_high: masked, f(r) = 0 */
#define SAO_FLAG_NONFINITE 3 /* log-ratio or advantage not finite: masked */
#define SAO_FLAG_NOT_ACTION 4/* loss_mask == 0 (prompt / observation token) */

/* Device-side error bits (checked mode), OR-ed into one word. */
#define SAO_DEVERR_TOKEN_ID 0x1u     /* some y[t] outside [0, V) */
#define SAO_DEVERR_CU_SEQLENS 0x2u   /* cu_seqlens not 0..N non-decreasing */
#define SAO_DEVERR_SCAN_TIMEOUT 0x4u /* advantage scan gave up waiting for a carry */
#define SAO_DEVERR_PIPE_TIMEOUT 0x8u /* a GEMM pipeline wait gave up */
#define SAO_DEVERR_CACHE_ROW 0x10u   /* cached backward: a row with grad != 0 the forward skipped */

/* Library version, major * 10000 + minor * 100 + patch. */
SAO_API int sao_version(void);

/* Message for the most recent non-OK status on the calling host thread. */
SAO_API const char *sao_last_error_string(void);

/* Checked mode (off by default): every call synchronises its stream, reads
 * and clears the device error word, and returns SAO_ERR_DEVICE_CHECK if it is
 * non-zero. Process-wide setting. */
SAO_API void sao_set_checked(int on);
SAO_API int sao_get_checked(void);

/* Upper bound on the bf16 dZ buffer of sao_token_logprobs_bwd (default
 * 4 GiB, at least 1 MiB). The backward never holds dZ for all N x V logits:
 * it works on blocks of rows times chunks of the vocabulary whose bf16 dZ fits
 * the budget (one block and one chunk when N x V does), choosing the split
 * with the least extra traffic (an fp32 dH accumulator read and written once
 * per extra vocabulary chunk; dW added to once per extra row block). Affects
 * sao_workspace_bytes. Process-wide. */
SAO_API void sao_set_dz_budget_bytes(size_t bytes);
/* The current bound (bytes) set by sao_set_dz_budget_bytes or the default. */
SAO_API size_t sao_get_dz_budget_bytes(void);

/* Tiling of the bf16 tensor-core GEMMs (process-wide; default 0). on = 1:
 * CTA pairs, clusters of 2 CTAs sharing each tcgen05.mma.cta_group::2 of
 * M = 256 (each CTA loads its own 128 rows of A and half of the B tile); on =
 * 0: single CTAs with M = 128 MMAs. Results agree to within the fp32
 * accumulation order. On one GB300 under its power cap the pairs do about 3 %
 * more work per SM clock but run at a lower clock, and the moe step takes
 * 2.5 % longer, hence the default. Affects later calls only. */
SAO_API void sao_set_cta_pairs(int on);
SAO_API int sao_get_cta_pairs(void);

/*
 * Test hooks of the advantage scan (process-wide; defaults restored by
 * (0, 0)): every look-back wait gives up after wait_ns nanoseconds (0: the
 * default 2 s; longer values are capped at it), and the scan's top
 * skip_chunks chunks (of 1024, 2048 or 4096 tokens, chosen from N) are never
 * processed, so the chunks below them
 * wait for a carry that never comes. Failure-detection tests use them to make
 * the bounded wait run out: the call still completes, the context stays
 * usable, and checked mode reports SAO_DEVERR_SCAN_TIMEOUT. Not for
 * production use (the skipped chunks' outputs are left unwritten).
 */
SAO_API void sao_debug_set_scan_hooks(uint64_t wait_ns, int32_t skip_chunks);

/* Workspace bytes that every entry point needs for N tokens, hidden size h,
 * vocabulary V and dtype dt (pass h = V = 0 when only the O(N) calls are
 * used). Returns 0 for invalid sizes. */
SAO_API size_t sao_workspace_bytes(int64_t N, int32_t h, int32_t V, sao_dtype dt);

/*
 * Eq. 1-2: logp[t] = z[t, y[t]] - lse[t], z = H W^T, lse[t] = log sum_v e^z[t,v].
 *   H        [N, h] dt, row-major          W  [V, h] dt, row-major
 *   y        [N] int32 in [0, V)           row_mask [N] uint8 or NULL: rows
 *            with row_mask[t] == 0 are not computed and get logp = lse = 0
 *   logp,lse [N] fp32 outputs (lse is kept for the backward)
 * Sizes: N >= 0; 1 <= V; h >= 1; for bf16, h % 8 == 0 (TMA row pitch).
 * A token id outside [0, V) yields logp = NaN (and SAO_DEVERR_TOKEN_ID).
 */
SAO_API sao_status sao_token_logprobs_fwd(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                  const uint8_t *row_mask, int64_t N, int32_t h, int32_t V,
                                  float *logp, float *lse, void *ws, size_t ws_bytes,
                                  sao_stream_t stream);

/*
 * Gradient of sum_t G[t] * logp[t] (G = grad_logp): with p = e^(z - lse),
 * dZ[t, v] = G[t] * (1[v == y[t]] - p[t, v]); dH = dZ W; dW = dZ^T H.
 *   lse       [N] fp32 from sao_token_logprobs_fwd on the same H, W, y
 *   grad_logp [N] fp32; rows with grad_logp == 0 contribute nothing
 *   dH        [N, h] dt output (overwritten)
 *   dW        [V, h] fp32 output; overwritten if accumulate_dW == 0, else
 *             the gradient is added to its contents
 */
SAO_API sao_status sao_token_logprobs_bwd(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                  const float *lse, const float *grad_logp, int64_t N, int32_t h,
                                  int32_t V, void *dH, float *dW, int accumulate_dW, void *ws,
                                  size_t ws_bytes, sao_stream_t stream);

/*
 * The same two calls with the forward's probabilities kept for the backward
 * (bf16 only), so the backward needs neither the logits nor dZ in memory.
 * For every row it computes, the forward takes a shift kappa = z[t, y] + 20
 * (the sampled token's logit, from a pre-pass) and stores e[t, v] = exp(z[t,
 * v] - kappa) in bf16; once lse is known, the entry at v = y becomes e[t, y] -
 * exp(lse - kappa). Then dZ[t, .] = -G[t] exp(kappa - lse[t]) e[t, .], and the
 * backward is two GEMMs on e: dH = (e W) scaled per row, dW = e^T (s H). A row
 * with some z[t, v] more than 60 above z[t, y] (p_y below e^-60) would
 * overflow that range: the forward flags it (its lse and log-prob are still
 * exact) and the backward recomputes that row's logits. The results match
 * sao_token_logprobs_fwd / _bwd within the bf16 rounding of e and of s H.
 *   cache        caller-owned device buffer of sao_logprob_cache_bytes(N, V)
 *                bytes (about 2 N V bytes), 256-byte aligned; written by the
 *                forward, read (not modified) by the backward, which must get
 *                the same H, W, y, N, V and the forward's lse
 * A backward row with grad_logp != 0 that the forward skipped (row_mask 0)
 * has no stored probabilities: it contributes nothing and raises
 * SAO_DEVERR_CACHE_ROW. Other arguments as the uncached calls; SAO_F32 gives
 * SAO_ERR_UNSUPPORTED.
 */
SAO_API size_t sao_logprob_cache_bytes(int64_t N, int32_t V);
SAO_API sao_status sao_token_logprobs_fwd_cached(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                                 const uint8_t *row_mask, int64_t N, int32_t h, int32_t V,
                                                 float *logp, float *lse, void *cache, size_t cache_bytes, void *ws,
                                                 size_t ws_bytes, sao_stream_t stream);
SAO_API sao_status sao_token_logprobs_bwd_cached(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                                 const float *lse, const float *grad_logp, int64_t N, int32_t h,
                                                 int32_t V, void *dH, float *dW, int accumulate_dW,
                                                 const void *cache, size_t cache_bytes, void *ws, size_t ws_bytes,
                                                 sao_stream_t stream);

/*
 * Skip-observation GAE (Preliminaries; §3.2 Eq. 4-5; §4.1). For trajectory b
 * (tokens cu_seqlens[b] .. cu_seqlens[b+1]-1) only action tokens
 * (loss_mask == 1) take part; the Bellman successor of an action token is the
 * next action token of the same trajectory, skipping observation tokens; the
 * value after the last action token is 0 and rewards[b] is the reward of the
 * last action token. delta_j = r_j + gamma V_next - V_j,
 * A_j = delta_j + gamma lambda_b A_next, ret_j = GAE(lambda_critic)_j + V_j.
 * lambda_b = lambda_policy, or 1 - 1/(alpha * L_b) clamped to [0,1] when
 * len_adaptive_alpha = alpha > 0 (L_b = number of action tokens of b).
 * Non-action tokens get adv = ret = 0. Computed in double-float (about 48
 * significant bits) and rounded to fp32.
 *   values [N] fp32, rewards [B] fp32, loss_mask [N] uint8,
 *   cu_seqlens [B+1] int32 with 0 = cu[0] <= ... <= cu[B] = N
 *   adv, ret [N] fp32 outputs
 * Scalars: 0 <= gamma, lambda_policy, lambda_critic <= 1.
 * Arrays that start 16-byte aligned move by TMA tensor copies; other
 * alignments are staged element by element (same results, slower).
 * The scan keeps each chunk's values in TMEM between its two passes: while it
 * runs, each SM's 512 TMEM columns are held by its CTAs, so a kernel on
 * another stream that allocates TMEM on the same SM waits for them (and the
 * scan waits for such a kernel's columns); neither depends on the other's
 * progress, so the wait always ends.
 */
SAO_API sao_status sao_advantages(const float *values, const float *rewards, const uint8_t *loss_mask,
                          const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma,
                          float lambda_policy, float lambda_critic, float len_adaptive_alpha,
                          float *adv, float *ret, void *ws, size_t ws_bytes, sao_stream_t stream);

/* Step value definitions of sao_step_advantages (App. A.1). */
#define SAO_STEP_AVERAGE 0 /* V(S) = mean of the step's token values; every step token is a value-loss token */
#define SAO_STEP_LAST 1    /* V(S) = value of the step's last token; only that token is a value-loss token */

/*
 * Step-level GAE (App. A.1, "RL with Agentic Step as Action"). A step is one
 * conversation turn: a maximal run of action tokens (loss_mask == 1) inside a
 * trajectory. With V(S_i) per `mode`, the terminal reward on the last step and
 * the step value after the last step 0: delta_i = r_i + gamma V(S_{i+1}) -
 * V(S_i), A_i = delta_i + gamma lambda A_{i+1} where lambda = lambda_policy,
 * or 1 - 1/(alpha * number of steps) clamped to [0,1] when
 * len_adaptive_alpha = alpha > 0 (the length-adaptive rule counted in steps).
 * Every token of step i receives adv = A_i and ret = GAE(lambda_critic)_i +
 * V(S_i); other tokens get 0. value_mask (nullable, [N] uint8) marks the
 * tokens the value loss keeps: all step tokens (SAO_STEP_AVERAGE) or the last
 * token of each step (SAO_STEP_LAST). Per-step sums are compensated fp32
 * pairs and the step recursion runs in double-float (about 48 bits each; the
 * fp64 pipe is not used), then each result is rounded once to fp32.
 * Arguments otherwise as sao_advantages; workspace from sao_workspace_bytes.
 */
SAO_API sao_status sao_step_advantages(const float *values, const float *rewards, const uint8_t *loss_mask,
                                       const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma,
                                       float lambda_policy, float lambda_critic, float len_adaptive_alpha, int mode,
                                       float *adv, float *ret, uint8_t *value_mask, void *ws, size_t ws_bytes,
                                       sao_stream_t stream);

/* Normalisation of sao_clip_loss_fwd/bwd (Preliminaries, unified objective). */
#define SAO_NORM_TOKEN 0    /* mean over all action tokens of the batch */
#define SAO_NORM_SEQUENCE 1 /* 1/|y| mean inside each trajectory, then the mean over trajectories */

/*
 * Clipped surrogate of the Preliminaries' unified objective with asymmetric
 * ("clip-higher") bounds: the loss of the paper's PPO/GRPO comparison arms
 * (§4.2; "GRPO w/ DIS" passes rollout log-probs as old_logp). With
 * r_t = exp(logp_t - old_logp_t):
 *   loss = -sum_t w_t min(r_t adv_t, clip(r_t, 1 - eps_low, 1 + eps_high) adv_t)
 * over action tokens, w_t = 1/(action tokens) for SAO_NORM_TOKEN, or
 * 1/(|y_b| * trajectories with an action token) for SAO_NORM_SEQUENCE. A token
 * is clipped when the min takes the clipped term strictly (adv > 0 and
 * r > 1 + eps_high: flag 2; adv < 0 and r < 1 - eps_low: flag 1), decided in
 * fp32; clipped tokens have coef = 0, others coef = d loss / d logp =
 * -w_t r_t adv_t. Non-finite tokens: flag 3, masked. counts = {n_action,
 * n_clip_low, n_clip_high, n_nonfinite}. coef and flags may be NULL.
 * cu_seqlens [B+1] as for sao_advantages (used by both normalisations).
 */
SAO_API sao_status sao_clip_loss_fwd(const float *logp, const float *old_logp, const float *adv,
                                     const uint8_t *loss_mask, const int32_t *cu_seqlens, int32_t B, int64_t N,
                                     float eps_low, float eps_high, int norm, float *loss, float *coef,
                                     uint8_t *flags, int64_t *counts, void *ws, size_t ws_bytes, sao_stream_t stream);

/* grad_logp[t] = grad_loss[0] * coef[t] of sao_clip_loss_fwd, recomputed. */
SAO_API sao_status sao_clip_loss_bwd(const float *logp, const float *old_logp, const float *adv,
                                     const uint8_t *loss_mask, const int32_t *cu_seqlens, int32_t B, int64_t N,
                                     float eps_low, float eps_high, int norm, const float *grad_loss,
                                     float *grad_logp, void *ws, size_t ws_bytes, sao_stream_t stream);

/*
 * GRPO's group-normalised advantage (Preliminaries): for trajectory b in
 * group g = group_ids[b], A_b = (R_b - mean_g R) / sqrt(var_g R + eps_stab)
 * (population variance over the group's trajectories: sums in compensated
 * fp32, about 48 bits, the final moments in fp64), broadcast to b's
 * action tokens; every other token gets 0. Cost O(B^2 / SMs) for the group
 * statistics (deterministic), then O(N).
 */
SAO_API sao_status sao_group_advantages(const float *rewards, const int32_t *group_ids, int32_t B,
                                        const uint8_t *loss_mask, const int32_t *cu_seqlens, int64_t N,
                                        float eps_stab, float *adv, void *ws, size_t ws_bytes, sao_stream_t stream);

/*
 * Running-mean reward baseline, the single-rollout alternative to a value
 * model in the ablations (§4.3: window of the 8 most recent rewards of each
 * prompt; §4.5: one window of the 128 most recent rewards, i.e. one prompt
 * id for all). Trajectories are taken in batch order: the baseline of b is
 * the mean of the at most `window` most recent rewards recorded for prompt
 * prompt_ids[b] before b (0 if none), A_b = R_b - baseline is written to b's
 * action tokens (0 elsewhere), then R_b enters that prompt's window.
 *   history [num_prompts, window] fp32 and seen [num_prompts] int64: the
 *   windows (ring buffers indexed by seen % window) and the number of rewards
 *   recorded per prompt; caller-owned device state, updated in place (zero
 *   both before the first batch). prompt_ids in [0, num_prompts); a
 *   trajectory with an id outside that range gets advantage 0 and is not
 *   recorded.
 */
SAO_API sao_status sao_running_mean_advantages(const float *rewards, const int32_t *prompt_ids, int32_t B,
                                               int32_t num_prompts, float *history, int64_t *seen, int32_t window,
                                               const uint8_t *loss_mask, const int32_t *cu_seqlens, int64_t N,
                                               float *adv, void *ws, size_t ws_bytes, sao_stream_t stream);

/* Extra per-token flag values written by sao_decoupled_loss_fwd. */
#define SAO_FLAG_MISMATCH_LOW 5  /* w = pi_old / pi_rollout <= w_low: masked */
#define SAO_FLAG_MISMATCH_HIGH 6 /* w >= w_high: masked */

/*
 * Decoupled three-policy objective, the mechanism that DIS simplifies (§3.1:
 * pi_theta / pi_old corrects staleness, pi_old / pi_rollout the training /
 * rollout mismatch, and tokens whose mismatch leaves a band are masked). With
 *   r_t = exp(logp_t - prox_logp_t)          (pi_theta / pi_old)
 *   w_t = exp(prox_logp_t - rollout_logp_t)  (pi_old / pi_rollout)
 * a token is kept when it is an action token, both log-ratios and adv_t are
 * finite and w_low < w_t < w_high (strict); then
 *   loss = -(1/n) sum_t w_t min(r_t adv_t, clip(r_t, 1 - eps_low, 1 + eps_high) adv_t)
 * with n = n_norm if n_norm > 0, else the number of action tokens. w is a
 * detached coefficient: coef_t = d loss / d logp_t = -w_t r_t adv_t / n when
 * the min keeps r_t adv_t (flag 0), and 0 when it is clipped (flag 1: adv < 0
 * and r < 1 - eps_low; flag 2: adv > 0 and r > 1 + eps_high) or the token is
 * masked (flags 3-6). Decisions are taken in fp32, the band before the clip.
 *   logp, prox_logp, rollout_logp, adv [N] fp32; loss_mask [N] uint8
 *   loss [1] fp32, coef [N] fp32 (nullable), flags [N] uint8 (nullable)
 *   counts [6] int64 = {n_action, n_clip_low, n_clip_high, n_nonfinite,
 *                       n_mismatch_low, n_mismatch_high}
 * Scalars: eps_low, eps_high >= 0; 0 <= w_low < w_high (w_high may be +inf).
 * Workspace from sao_workspace_bytes. Deterministic (fixed-order reductions).
 */
SAO_API sao_status sao_decoupled_loss_fwd(const float *logp, const float *prox_logp, const float *rollout_logp,
                                          const float *adv, const uint8_t *loss_mask, int64_t N, float eps_low,
                                          float eps_high, float w_low, float w_high, int64_t n_norm, float *loss,
                                          float *coef, uint8_t *flags, int64_t *counts, void *ws, size_t ws_bytes,
                                          sao_stream_t stream);

/* grad_logp[t] = grad_loss[0] * coef[t] of sao_decoupled_loss_fwd, recomputed
 * from the inputs (stateless); grad_loss is a device scalar. */
SAO_API sao_status sao_decoupled_loss_bwd(const float *logp, const float *prox_logp, const float *rollout_logp,
                                          const float *adv, const uint8_t *loss_mask, int64_t N, float eps_low,
                                          float eps_high, float w_low, float w_high, int64_t n_norm,
                                          const float *grad_loss, float *grad_logp, void *ws, size_t ws_bytes,
                                          sao_stream_t stream);

/*
 * sao_advantages without a workspace argument, for callers that cannot
 * allocate device memory: a host library that is handed only data pointers
 * and a stream by another framework and has no allocator of its own, or a
 * process that reserves all device memory at start-up and forbids later
 * allocations (cudaMalloc also synchronises the whole device, which a
 * latency-critical caller cannot afford). The paper has no counterpart to
 * this entry point; it computes exactly what sao_advantages computes.
 *
 * Scratch: a fixed 16 MiB array inside this library's device image, present on
 * every GPU that loads the library until the process exits. It bounds the
 * sizes: about 200 bytes per 1024 tokens plus 36 bytes per trajectory must
 * fit (for example 2^25 tokens with up to 65,536 trajectories); larger
 * inputs return SAO_ERR_SHAPE with the bytes needed. Nothing is allocated
 * and nothing is freed.
 * Each call made outside stream capture looks up the array's device address
 * (with the calling thread's current device) and remembers it for that
 * device, so a device reset or a new primary context is picked up; a call
 * under stream capture uses the remembered address and returns
 * SAO_ERR_INVALID_ARG if no call on that device came before the capture.
 * Every call on a device shares the one array, so calls that overlap
 * on the GPU (two streams, or two threads) race and corrupt each other's
 * results; serialise them. Each call clears the parts of the array that must
 * start at zero, so stale contents from a previous call do no harm.
 */
SAO_API sao_status sao_advantages_noalloc(const float *values, const float *rewards, const uint8_t *loss_mask,
                                          const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma,
                                          float lambda_policy, float lambda_critic, float len_adaptive_alpha,
                                          float *adv, float *ret, sao_stream_t stream);

/*
 * Eq. 1-3 (§3.1). r_t = exp(logp_t - old_logp_t); a token is kept iff it is an
 * action token, its log-ratio and advantage are finite and
 * 1 - eps_low < r_t < 1 + eps_high (strict; decided in fp32). With n = n_norm
 * if n_norm > 0, else the number of action tokens:
 *   loss    = -(1/n) sum_{kept t} r_t adv_t            [1] fp32 output
 *   coef[t] = d loss / d logp_t = -r_t adv_t / n (kept), 0 otherwise (f(r) is
 *             a detached coefficient)                   [N] fp32 output
 *   flags[t]  SAO_FLAG_* value                          [N] uint8 output
 *   counts  = {n_action, n_low, n_high, n_nonfinite}    [4] int64 output
 * coef and flags may be NULL. The reductions are deterministic.
 * Scalars: eps_low >= 0 (eps_low >= 1 disables the lower bound), eps_high >= 0.
 */
SAO_API sao_status sao_policy_loss_fwd(const float *logp, const float *old_logp, const float *adv,
                               const uint8_t *loss_mask, int64_t N, float eps_low, float eps_high,
                               int64_t n_norm, float *loss, float *coef, uint8_t *flags,
                               int64_t *counts, void *ws, size_t ws_bytes, sao_stream_t stream);

/*
 * grad_logp[t] = grad_loss[0] * coef[t], with coef recomputed from the same
 * inputs as sao_policy_loss_fwd (stateless). grad_loss is a device scalar.
 */
SAO_API sao_status sao_policy_loss_bwd(const float *logp, const float *old_logp, const float *adv,
                               const uint8_t *loss_mask, int64_t N, float eps_low, float eps_high,
                               int64_t n_norm, const float *grad_loss, float *grad_logp, void *ws,
                               size_t ws_bytes, sao_stream_t stream);

/*
 * Value loss (Preliminaries, PPO): over the action tokens, with n = n_norm if
 * n_norm > 0, else the number of action tokens,
 *   loss = (1/n) sum_t (V_t - ret_t)^2           [1] fp32 output
 *   grad_values[t] = 2 (V_t - ret_t) / n, 0 on non-action tokens   [N] fp32
 *   ev_sums = {sum (R-V), sum (R-V)^2, sum R, sum R^2} over action tokens
 *             ([4] fp64, may be NULL), from which explained variance
 *             EV = 1 - Var(R - V) / Var(R) (§4.4) follows.
 * n_norm is the normaliser shared by data-parallel ranks (the action tokens
 * of the whole batch), as for the policy loss: the ranks' losses and
 * gradients then add up to those of the unsplit batch. With n_norm > 0 the
 * call makes one pass over the tokens; otherwise it counts them first.
 */
SAO_API sao_status sao_value_loss(const float *values, const float *ret, const uint8_t *loss_mask,
                          int64_t N, int64_t n_norm, float *loss, float *grad_values, double *ev_sums,
                          void *ws, size_t ws_bytes, sao_stream_t stream);

/*
 * Kernel timing for profiling. When enabled, every kernel the library
 * launches is bracketed by CUDA events on its stream; sao_profile_read
 * synchronises those events and returns, for up to `cap` kernel kinds, the
 * name (static string), the number of launches and the summed device
 * milliseconds since the last reset. Returns the number of kinds written.
 */
SAO_API void sao_profile_enable(int on);
SAO_API void sao_profile_reset(void);
SAO_API int sao_profile_read(const char **names, int64_t *launches, double *total_ms, int cap);

#ifdef __cplusplus
}
#endif

#endif /* SAO_H_ */
