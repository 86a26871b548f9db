// extern "C" entry points of libsao: argument checks, workspace carving and
// dispatch to the kernel launchers. See include/sao.h for the contract.
#include <math.h>
#include <stdint.h>

#include <atomic>

#include <nvtx3/nvToolsExt.h>

#include "logprobs_common.cuh"
#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {

static std::atomic<size_t> g_dz_budget{size_t(4) << 30};
void set_dz_budget(size_t bytes) { g_dz_budget.store(bytes < (size_t(1) << 20) ? (size_t(1) << 20) : bytes); }
size_t dz_budget() { return g_dz_budget.load(); }

static std::atomic<int> g_cta_pairs{0};
void set_cta_pairs(int on) { g_cta_pairs.store(on ? 1 : 0); }
int cta_group() { return g_cta_pairs.load() ? 2 : 1; }

static std::atomic<uint64_t> g_scan_wait_ns{kWaitLimitNs};
static std::atomic<int> g_scan_skip{0};
uint64_t scan_wait_ns() { return g_scan_wait_ns.load(); }
int scan_skip() { return g_scan_skip.load(); }

// O(N) kernels size their grids from N alone (deterministic on any device).
size_t on_ws_bytes(int64_t N) {
  size_t w = elementwise_ws_bytes(N, 0);
  const size_t g = gae_ws_bytes(N, N + 1);
  const size_t st = step_gae_ws_bytes(N, N + 1);
  const size_t bl = baselines_ws_bytes(N, N + 1);
  if (g > w) w = g;
  if (st > w) w = st;
  if (bl > w) w = bl;
  return w;
}

size_t logprobs_ws_bytes(int64_t N, int32_t h, int32_t V, sao_dtype dt) {
  if (h <= 0 || V <= 0) return 0;
  return dt == SAO_BF16 ? tc_ws_bytes(N, h, V) : simt_ws_bytes(N, h, V);
}

}  // namespace sao

using namespace sao;

namespace {

// An NVTX range around every entry point, so a profiler timeline shows the
// ABI calls with their kernels (header-only NVTX: no cost without a tool).
struct NvtxRange {
  explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange &) = delete;
  NvtxRange &operator=(const NvtxRange &) = delete;
};
#define SAO_RANGE() NvtxRange sao_nvtx_range_(__func__)

struct Ws {
  unsigned int *err;
  void *body;
  size_t body_bytes;
};

sao_status take_ws(void *ws, size_t ws_bytes, size_t need_body, Ws *out) {
  if (ws == nullptr) return fail(SAO_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(SAO_ERR_INVALID_ARG, "workspace is not 256-byte aligned");
  if (ws_bytes < kWsHeader + need_body)
    return fail(SAO_ERR_WORKSPACE, "workspace of %zu bytes, %zu needed", ws_bytes, kWsHeader + need_body);
  out->err = static_cast<unsigned int *>(ws);
  out->body = static_cast<char *>(ws) + kWsHeader;
  out->body_bytes = ws_bytes - kWsHeader;
  return SAO_OK;
}

bool bad_dtype(sao_dtype dt) { return dt != SAO_F32 && dt != SAO_BF16; }

sao_status check_logprob_shapes(sao_dtype dt, int64_t N, int32_t h, int32_t V) {
  if (bad_dtype(dt)) return fail(SAO_ERR_UNSUPPORTED, "unknown dtype %d", int(dt));
  if (N < 0 || N >= (int64_t(1) << 31)) return fail(SAO_ERR_SHAPE, "N = %lld out of range", (long long)N);
  if (h < 1 || V < 1) return fail(SAO_ERR_SHAPE, "h = %d and V = %d must be >= 1", h, V);
  if (dt == SAO_BF16 && (h % 8) != 0) return fail(SAO_ERR_SHAPE, "bf16 needs h %% 8 == 0 (h = %d)", h);
  return SAO_OK;
}

sao_status check_tc_device(sao_dtype dt) {
  if (dt != SAO_BF16) return SAO_OK;
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  if (di.cc_major != 10 || di.cc_minor != 3)
    return fail(SAO_ERR_UNSUPPORTED, "the bf16 tensor-core path needs an sm_103 device (found sm_%d%d)",
                di.cc_major, di.cc_minor);
  return SAO_OK;
}

}  // namespace

extern "C" {

int sao_version(void) { return 100; }

const char *sao_last_error_string(void) { return last_error(); }

void sao_set_checked(int on) { set_checked(on); }
int sao_get_checked(void) { return checked_mode() ? 1 : 0; }

void sao_set_dz_budget_bytes(size_t bytes) { set_dz_budget(bytes); }
size_t sao_get_dz_budget_bytes(void) { return dz_budget(); }

void sao_set_cta_pairs(int on) { set_cta_pairs(on); }
int sao_get_cta_pairs(void) { return cta_group() == 2 ? 1 : 0; }

void sao_debug_set_scan_hooks(uint64_t wait_ns, int32_t skip_chunks) {
  g_scan_wait_ns.store(wait_ns == 0 ? kWaitLimitNs : (wait_ns > kWaitLimitNs ? kWaitLimitNs : wait_ns));
  g_scan_skip.store(skip_chunks > 0 ? skip_chunks : 0);
}

size_t sao_workspace_bytes(int64_t N, int32_t h, int32_t V, sao_dtype dt) {
  if (N < 0 || h < 0 || V < 0 || bad_dtype(dt)) return 0;
  size_t body = on_ws_bytes(N);
  const size_t lp = logprobs_ws_bytes(N, h, V, dt);
  if (lp > body) body = lp;
  return kWsHeader + body;
}

sao_status sao_token_logprobs_fwd(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                  const uint8_t *row_mask, int64_t N, int32_t h, int32_t V, float *logp,
                                  float *lse, void *ws, size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_logprob_shapes(dt, N, h, V));
  if (N == 0) return SAO_OK;
  if (!H || !W || !y || !logp || !lse) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  SAO_TRY(check_tc_device(dt));
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, logprobs_ws_bytes(N, h, V, dt), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  if (dt == SAO_BF16)
    SAO_TRY(tc_fwd(H, W, y, row_mask, N, h, V, logp, lse, w.err, w.body, w.body_bytes, nullptr, s));
  else
    SAO_TRY(simt_fwd(static_cast<const float *>(H), static_cast<const float *>(W), y, row_mask, N, h, V, logp,
                     lse, w.err, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_token_logprobs_bwd(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                  const float *lse, const float *grad_logp, int64_t N, int32_t h, int32_t V,
                                  void *dH, float *dW, int accumulate_dW, void *ws, size_t ws_bytes,
                                  sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_logprob_shapes(dt, N, h, V));
  if (!W || !dW) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (N == 0) {
    if (!accumulate_dW) SAO_CUDA_TRY(cudaMemsetAsync(dW, 0, sizeof(float) * size_t(V) * size_t(h), s));
    return SAO_OK;
  }
  if (!H || !y || !lse || !grad_logp || !dH) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  SAO_TRY(check_tc_device(dt));
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, logprobs_ws_bytes(N, h, V, dt), &w));
  SAO_TRY(begin_call(ws, s));
  if (dt == SAO_BF16)
    SAO_TRY(tc_bwd(H, W, y, lse, grad_logp, N, h, V, dH, dW, accumulate_dW, w.err, w.body, w.body_bytes, nullptr,
                   s));
  else
    SAO_TRY(simt_bwd(static_cast<const float *>(H), static_cast<const float *>(W), y, lse, grad_logp, N, h, V,
                     static_cast<float *>(dH), dW, accumulate_dW, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

size_t sao_logprob_cache_bytes(int64_t N, int32_t V) {
  if (N <= 0 || V <= 0) return 0;
  return logprob_cache_view(nullptr, N, V).bytes;
}

// The cache must hold sao_logprob_cache_bytes(N, V) bytes at a 256-byte
// aligned address (its parts are TMA operands and 16-byte vector streams).
static sao_status take_cache(const void *cache, size_t cache_bytes, int64_t N, int32_t V, LogprobCache *out) {
  if (!cache) return fail(SAO_ERR_INVALID_ARG, "NULL probability cache");
  if ((reinterpret_cast<uintptr_t>(cache) & 255u) != 0)
    return fail(SAO_ERR_INVALID_ARG, "probability cache not 256-byte aligned");
  *out = logprob_cache_view(const_cast<void *>(cache), N, V);
  if (cache_bytes < out->bytes)
    return fail(SAO_ERR_WORKSPACE, "probability cache too small: %zu bytes, need %zu", cache_bytes, out->bytes);
  return SAO_OK;
}

sao_status sao_token_logprobs_fwd_cached(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                         const uint8_t *row_mask, int64_t N, int32_t h, int32_t V, float *logp,
                                         float *lse, void *cache, size_t cache_bytes, void *ws, size_t ws_bytes,
                                         sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_logprob_shapes(dt, N, h, V));
  if (dt != SAO_BF16) return fail(SAO_ERR_UNSUPPORTED, "the probability cache is for bf16 only");
  if (N == 0) return SAO_OK;
  if (!H || !W || !y || !logp || !lse) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  SAO_TRY(check_tc_device(dt));
  LogprobCache k;
  SAO_TRY(take_cache(cache, cache_bytes, N, V, &k));
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, logprobs_ws_bytes(N, h, V, dt), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(tc_fwd(H, W, y, row_mask, N, h, V, logp, lse, w.err, w.body, w.body_bytes, &k, s));
  return finish_call(ws, s);
}

sao_status sao_token_logprobs_bwd_cached(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                                         const float *lse, const float *grad_logp, int64_t N, int32_t h, int32_t V,
                                         void *dH, float *dW, int accumulate_dW, const void *cache,
                                         size_t cache_bytes, void *ws, size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_logprob_shapes(dt, N, h, V));
  if (dt != SAO_BF16) return fail(SAO_ERR_UNSUPPORTED, "the probability cache is for bf16 only");
  if (!W || !dW) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (N == 0) {
    if (!accumulate_dW) SAO_CUDA_TRY(cudaMemsetAsync(dW, 0, sizeof(float) * size_t(V) * size_t(h), s));
    return SAO_OK;
  }
  if (!H || !y || !lse || !grad_logp || !dH) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  SAO_TRY(check_tc_device(dt));
  LogprobCache k;
  SAO_TRY(take_cache(cache, cache_bytes, N, V, &k));
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, logprobs_ws_bytes(N, h, V, dt), &w));
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(tc_bwd(H, W, y, lse, grad_logp, N, h, V, dH, dW, accumulate_dW, w.err, w.body, w.body_bytes, &k, s));
  return finish_call(ws, s);
}

sao_status sao_advantages(const float *values, const float *rewards, const uint8_t *loss_mask,
                          const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma, float lambda_policy,
                          float lambda_critic, float len_adaptive_alpha, float *adv, float *ret, void *ws,
                          size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0 || N >= (int64_t(1) << 31)) return fail(SAO_ERR_SHAPE, "N = %lld out of range", (long long)N);
  if (B < 0) return fail(SAO_ERR_SHAPE, "B = %d < 0", B);
  if (N > 0 && B == 0) return fail(SAO_ERR_SHAPE, "N > 0 tokens need at least one trajectory");
  if (!(gamma >= 0.f && gamma <= 1.f) || !(lambda_policy >= 0.f && lambda_policy <= 1.f) ||
      !(lambda_critic >= 0.f && lambda_critic <= 1.f) || !isfinite(len_adaptive_alpha))
    return fail(SAO_ERR_INVALID_ARG, "gamma and lambdas must lie in [0, 1] and alpha be finite");
  if (N == 0) return SAO_OK;
  if (!values || !rewards || !loss_mask || !cu_seqlens || !adv || !ret)
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, gae_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(gae_launch(values, rewards, loss_mask, cu_seqlens, B, N, gamma, lambda_policy, lambda_critic,
                     len_adaptive_alpha, adv, ret, w.err, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_step_advantages(const float *values, const float *rewards, const uint8_t *loss_mask,
                               const int32_t *cu_seqlens, int32_t B, int64_t N, float gamma, float lambda_policy,
                               float lambda_critic, float len_adaptive_alpha, int mode, float *adv, float *ret,
                               uint8_t *value_mask, void *ws, size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0 || N >= (int64_t(1) << 31)) return fail(SAO_ERR_SHAPE, "N = %lld out of range", (long long)N);
  if (B < 0) return fail(SAO_ERR_SHAPE, "B = %d < 0", B);
  if (N > 0 && B == 0) return fail(SAO_ERR_SHAPE, "N > 0 tokens need at least one trajectory");
  if (mode != SAO_STEP_AVERAGE && mode != SAO_STEP_LAST) return fail(SAO_ERR_INVALID_ARG, "unknown step mode %d", mode);
  if (!(gamma >= 0.f && gamma <= 1.f) || !(lambda_policy >= 0.f && lambda_policy <= 1.f) ||
      !(lambda_critic >= 0.f && lambda_critic <= 1.f) || !isfinite(len_adaptive_alpha))
    return fail(SAO_ERR_INVALID_ARG, "gamma and lambdas must lie in [0, 1] and alpha be finite");
  if (N == 0) return SAO_OK;
  if (!values || !rewards || !loss_mask || !cu_seqlens || !adv || !ret)
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, step_gae_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(step_gae_launch(values, rewards, loss_mask, cu_seqlens, B, N, gamma, lambda_policy, lambda_critic,
                          len_adaptive_alpha, mode, adv, ret, value_mask, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

static sao_status check_eps(float eps_low, float eps_high) {
  if (!(eps_low >= 0.f) || !(eps_high >= 0.f) || isnan(eps_low) || isnan(eps_high))
    return fail(SAO_ERR_INVALID_ARG, "clip bounds must be >= 0 (eps_low = %g, eps_high = %g)", eps_low, eps_high);
  return SAO_OK;
}

sao_status sao_policy_loss_fwd(const float *logp, const float *old_logp, const float *adv,
                               const uint8_t *loss_mask, int64_t N, float eps_low, float eps_high, int64_t n_norm,
                               float *loss, float *coef, uint8_t *flags, int64_t *counts, void *ws,
                               size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0) return fail(SAO_ERR_SHAPE, "N < 0");
  SAO_TRY(check_eps(eps_low, eps_high));
  if (!loss || !counts) return fail(SAO_ERR_INVALID_ARG, "NULL loss or counts");
  if (N > 0 && (!logp || !old_logp || !adv || !loss_mask)) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, elementwise_ws_bytes(N, 0), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(policy_loss_launch(logp, old_logp, adv, loss_mask, N, eps_low, eps_high, n_norm, loss, coef, flags,
                             counts, nullptr, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_policy_loss_bwd(const float *logp, const float *old_logp, const float *adv,
                               const uint8_t *loss_mask, int64_t N, float eps_low, float eps_high, int64_t n_norm,
                               const float *grad_loss, float *grad_logp, void *ws, size_t ws_bytes,
                               sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0) return fail(SAO_ERR_SHAPE, "N < 0");
  SAO_TRY(check_eps(eps_low, eps_high));
  if (N == 0) return SAO_OK;
  if (!logp || !old_logp || !adv || !loss_mask || !grad_loss || !grad_logp)
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, elementwise_ws_bytes(N, 0), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(policy_loss_launch(logp, old_logp, adv, loss_mask, N, eps_low, eps_high, n_norm, nullptr, grad_logp,
                             nullptr, nullptr, grad_loss, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

static sao_status check_band(float w_low, float w_high) {
  if (!(w_low >= 0.f) || !(w_high > w_low) || isnan(w_low) || isnan(w_high))
    return fail(SAO_ERR_INVALID_ARG, "mismatch band needs 0 <= w_low < w_high (w_low = %g, w_high = %g)", w_low,
                w_high);
  return SAO_OK;
}

sao_status sao_decoupled_loss_fwd(const float *logp, const float *prox_logp, const float *rollout_logp,
                                  const float *adv, const uint8_t *loss_mask, int64_t N, float eps_low,
                                  float eps_high, float w_low, float w_high, int64_t n_norm, float *loss,
                                  float *coef, uint8_t *flags, int64_t *counts, void *ws, size_t ws_bytes,
                                  sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0) return fail(SAO_ERR_SHAPE, "N < 0");
  SAO_TRY(check_eps(eps_low, eps_high));
  SAO_TRY(check_band(w_low, w_high));
  if (!loss || !counts) return fail(SAO_ERR_INVALID_ARG, "NULL loss or counts");
  if (N > 0 && (!logp || !prox_logp || !rollout_logp || !adv || !loss_mask))
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, elementwise_ws_bytes(N, 0), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(decoupled_loss_launch(logp, prox_logp, rollout_logp, adv, loss_mask, N, eps_low, eps_high, w_low, w_high,
                                n_norm, loss, coef, flags, counts, nullptr, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_decoupled_loss_bwd(const float *logp, const float *prox_logp, const float *rollout_logp,
                                  const float *adv, const uint8_t *loss_mask, int64_t N, float eps_low,
                                  float eps_high, float w_low, float w_high, int64_t n_norm, const float *grad_loss,
                                  float *grad_logp, void *ws, size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0) return fail(SAO_ERR_SHAPE, "N < 0");
  SAO_TRY(check_eps(eps_low, eps_high));
  SAO_TRY(check_band(w_low, w_high));
  if (N == 0) return SAO_OK;
  if (!logp || !prox_logp || !rollout_logp || !adv || !loss_mask || !grad_loss || !grad_logp)
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, elementwise_ws_bytes(N, 0), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(decoupled_loss_launch(logp, prox_logp, rollout_logp, adv, loss_mask, N, eps_low, eps_high, w_low, w_high,
                                n_norm, nullptr, grad_logp, nullptr, nullptr, grad_loss, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_value_loss(const float *values, const float *ret, const uint8_t *loss_mask, int64_t N, int64_t n_norm,
                          float *loss, float *grad_values, double *ev_sums, void *ws, size_t ws_bytes,
                          sao_stream_t stream) {
  SAO_RANGE();
  if (N < 0) return fail(SAO_ERR_SHAPE, "N < 0");
  if (!loss) return fail(SAO_ERR_INVALID_ARG, "NULL loss");
  if (N > 0 && (!values || !ret || !loss_mask || !grad_values)) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, elementwise_ws_bytes(N, 0), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(value_loss_launch(values, ret, loss_mask, N, n_norm, loss, grad_values, ev_sums, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

static sao_status check_traj(int32_t B, int64_t N, const int32_t *cu) {
  if (N < 0 || N >= (int64_t(1) << 31)) return fail(SAO_ERR_SHAPE, "N = %lld out of range", (long long)N);
  if (B < 0) return fail(SAO_ERR_SHAPE, "B = %d < 0", B);
  if (N > 0 && (B == 0 || !cu)) return fail(SAO_ERR_SHAPE, "N > 0 tokens need at least one trajectory");
  return SAO_OK;
}

sao_status sao_clip_loss_fwd(const float *logp, const float *old_logp, const float *adv, const uint8_t *loss_mask,
                             const int32_t *cu_seqlens, int32_t B, int64_t N, float eps_low, float eps_high, int norm,
                             float *loss, float *coef, uint8_t *flags, int64_t *counts, void *ws, size_t ws_bytes,
                             sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_traj(B, N, cu_seqlens));
  SAO_TRY(check_eps(eps_low, eps_high));
  if (norm != SAO_NORM_TOKEN && norm != SAO_NORM_SEQUENCE) return fail(SAO_ERR_INVALID_ARG, "unknown norm %d", norm);
  if (!loss || !counts) return fail(SAO_ERR_INVALID_ARG, "NULL loss or counts");
  if (N > 0 && (!logp || !old_logp || !adv || !loss_mask)) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, baselines_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(clip_loss_launch(logp, old_logp, adv, loss_mask, cu_seqlens, B, N, eps_low, eps_high, norm, loss, coef,
                           flags, counts, nullptr, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_clip_loss_bwd(const float *logp, const float *old_logp, const float *adv, const uint8_t *loss_mask,
                             const int32_t *cu_seqlens, int32_t B, int64_t N, float eps_low, float eps_high, int norm,
                             const float *grad_loss, float *grad_logp, void *ws, size_t ws_bytes,
                             sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_traj(B, N, cu_seqlens));
  SAO_TRY(check_eps(eps_low, eps_high));
  if (norm != SAO_NORM_TOKEN && norm != SAO_NORM_SEQUENCE) return fail(SAO_ERR_INVALID_ARG, "unknown norm %d", norm);
  if (N == 0) return SAO_OK;
  if (!logp || !old_logp || !adv || !loss_mask || !grad_loss || !grad_logp)
    return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, baselines_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(clip_loss_launch(logp, old_logp, adv, loss_mask, cu_seqlens, B, N, eps_low, eps_high, norm, nullptr,
                           grad_logp, nullptr, nullptr, grad_loss, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_group_advantages(const float *rewards, const int32_t *group_ids, int32_t B, const uint8_t *loss_mask,
                                const int32_t *cu_seqlens, int64_t N, float eps_stab, float *adv, void *ws,
                                size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_traj(B, N, cu_seqlens));
  if (!(eps_stab >= 0.f) || !isfinite(eps_stab)) return fail(SAO_ERR_INVALID_ARG, "eps_stab must be >= 0");
  if (N == 0) return SAO_OK;
  if (!rewards || !group_ids || !loss_mask || !adv) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, baselines_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(group_adv_launch(rewards, group_ids, B, loss_mask, cu_seqlens, N, eps_stab, adv, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

sao_status sao_running_mean_advantages(const float *rewards, const int32_t *prompt_ids, int32_t B,
                                       int32_t num_prompts, float *history, int64_t *seen, int32_t window,
                                       const uint8_t *loss_mask, const int32_t *cu_seqlens, int64_t N, float *adv,
                                       void *ws, size_t ws_bytes, sao_stream_t stream) {
  SAO_RANGE();
  SAO_TRY(check_traj(B, N, cu_seqlens));
  if (window < 1 || num_prompts < 1) return fail(SAO_ERR_INVALID_ARG, "window and num_prompts must be >= 1");
  if (B > 0 && (!rewards || !prompt_ids || !history || !seen)) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  if (N > 0 && (!loss_mask || !adv)) return fail(SAO_ERR_INVALID_ARG, "NULL array argument");
  Ws w;
  SAO_TRY(take_ws(ws, ws_bytes, baselines_ws_bytes(N, B), &w));
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  SAO_TRY(begin_call(ws, s));
  SAO_TRY(running_mean_launch(rewards, prompt_ids, B, num_prompts, history, seen, window, loss_mask, cu_seqlens, N,
                              adv, w.body, w.body_bytes, s));
  return finish_call(ws, s);
}

void sao_profile_enable(int on) { profile_enable(on); }
void sao_profile_reset(void) { profile_reset(); }
int sao_profile_read(const char **names, int64_t *launches, double *total_ms, int cap) {
  return profile_read(names, launches, total_ms, cap);
}

}  // extern "C"
