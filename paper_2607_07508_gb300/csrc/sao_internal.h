// Internal launcher interface between the C-ABI layer and the kernel files.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sao.h"

namespace sao {

__host__ __device__ inline bool aligned16_dev(const void *p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// elementwise.cu ------------------------------------------------------------
size_t elementwise_ws_bytes(int64_t N, int sm_count);
sao_status policy_loss_launch(const float *logp, const float *old, const float *adv, const uint8_t *m,
                              int64_t N, float eps_low, float eps_high, int64_t n_norm, float *loss,
                              float *coef, uint8_t *flags, int64_t *counts, const float *grad_loss,
                              void *ws_body, size_t body_bytes, cudaStream_t s);
sao_status value_loss_launch(const float *v, const float *ret, const uint8_t *m, int64_t N, int64_t n_norm, float *loss,
                             float *grad, double *ev, void *ws_body, size_t body_bytes, cudaStream_t s);
sao_status decoupled_loss_launch(const float *logp, const float *prox, const float *roll, const float *adv,
                                 const uint8_t *m, int64_t N, float eps_low, float eps_high, float w_low,
                                 float w_high, int64_t n_norm, float *loss, float *coef, uint8_t *flags,
                                 int64_t *counts, const float *grad_loss, void *ws_body, size_t body_bytes,
                                 cudaStream_t s);

// logprobs_tc.cu: the driver's tensor-map encoder (null when the driver has
// none), shared by every kernel that stages tiles with TMA
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

// gae.cu ----------------------------------------------------------------------
size_t gae_ws_bytes(int64_t N, int64_t B);
sao_status gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu,
                      int32_t B, int64_t N, float gamma, float lam, float lam_c, float alpha, float *adv,
                      float *ret, unsigned int *err, void *ws_body, size_t body_bytes, cudaStream_t s);

// step_gae.cu -----------------------------------------------------------------
size_t step_gae_ws_bytes(int64_t N, int64_t B);
sao_status step_gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu, int32_t B,
                           int64_t N, float gamma, float lam, float lam_c, float alpha, int mode, float *adv,
                           float *ret, uint8_t *vmask, void *ws_body, size_t body_bytes, cudaStream_t s);

// baselines.cu ----------------------------------------------------------------
size_t baselines_ws_bytes(int64_t N, int64_t B);
sao_status clip_loss_launch(const float *logp, const float *old, const float *adv, const uint8_t *m, const int32_t *cu,
                            int32_t B, int64_t N, float eps_low, float eps_high, int norm, float *loss, float *coef,
                            uint8_t *flags, int64_t *counts, const float *grad_loss, void *ws_body,
                            size_t body_bytes, cudaStream_t s);
sao_status running_mean_launch(const float *rewards, const int32_t *pid, int32_t B, int32_t P, float *history,
                               int64_t *seen, int32_t window, const uint8_t *m, const int32_t *cu, int64_t N,
                               float *adv, void *ws_body, size_t body_bytes, cudaStream_t s);
sao_status group_adv_launch(const float *rewards, const int32_t *gid, int32_t B, const uint8_t *m, const int32_t *cu,
                            int64_t N, float eps, float *adv, void *ws_body, size_t body_bytes, cudaStream_t s);

// logprobs (tensor-core and fp32 paths) ----------------------------------------
size_t logprobs_ws_bytes(int64_t N, int32_t h, int32_t V, sao_dtype dt);
sao_status logprobs_fwd_launch(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                               const uint8_t *row_mask, int64_t N, int32_t h, int32_t V, float *logp,
                               float *lse, unsigned int *err, void *ws_body, size_t body_bytes,
                               cudaStream_t s);
sao_status logprobs_bwd_launch(const void *H, const void *W, sao_dtype dt, const int32_t *y,
                               const float *lse, const float *G, int64_t N, int32_t h, int32_t V,
                               void *dH, float *dW, int accumulate, unsigned int *err, void *ws_body,
                               size_t body_bytes, cudaStream_t s);

void set_dz_budget(size_t bytes);
size_t dz_budget();
// GEMM tiling of the tensor-core path: 1 = single CTAs, 2 = CTA pairs.
void set_cta_pairs(int on);
int cta_group();

// Test hooks of the advantage scan (see sao_debug_set_scan_hooks in sao.h).
uint64_t scan_wait_ns();
int scan_skip();

}  // namespace sao
