// Pieces shared by the fp32 and tensor-core log-prob paths.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/sao.h"

namespace sao {

// Merges per-(vocab tile, row) partials part[j * N + i] = (max_j, sumexp_j)
// into lse[row] = log sum_v e^z and logp[row] = zy[i] - lse[row], where i is
// the row itself, or pos[row] when the forward ran on compacted rows (pos < 0:
// a skipped row, logp = lse = 0). Rows with row_mask == 0 also get zeros.
// Token ids outside [0, V) give logp = NaN.
sao_status lse_merge_launch(const float2 *part, int nvt, const float *zy, const int32_t *y,
                            const uint8_t *row_mask, const int *pos, int64_t N, int32_t V, float *logp, float *lse,
                            unsigned int *err, cudaStream_t s);

size_t simt_ws_bytes(int64_t N, int32_t h, int32_t V);
sao_status simt_fwd(const float *H, const float *W, const int32_t *y, const uint8_t *row_mask, int64_t N,
                    int32_t h, int32_t V, float *logp, float *lse, unsigned int *err, void *ws, size_t ws_bytes,
                    cudaStream_t s);
sao_status simt_bwd(const float *H, const float *W, const int32_t *y, const float *lse, const float *G,
                    int64_t N, int32_t h, int32_t V, float *dH, float *dW, int accumulate, void *ws,
                    size_t ws_bytes, cudaStream_t s);

// The forward's stored probabilities (tensor-core path). For forward row f
// (token idx[f]) with shift kappa[f] = z[f, y] + kKappaOffset, where z[f, y]
// is the sampled token's logit from a pre-pass, e[f, v] = exp(z[f, v] -
// kappa[f]) in bf16, except at v = y, which holds e[f, y] - exp(lse - kappa)
// once the forward has lse. Then dZ[f, .] = -G exp(kappa - lse) e[f, .]: the
// backward is two GEMMs on e with a per-row scale. flag[f] marks a row where
// some z - kappa exceeded kFlagExponent (its stored values were clamped); the
// backward recomputes those rows' logits instead.
constexpr float kKappaOffset = 20.f;
constexpr float kFlagExponent = 40.f;
struct LogprobCache {
  __nv_bfloat16 *e;   // [rows, lde]
  int64_t lde, rows;
  int *idx;           // [N] forward row -> token
  int *pos;           // [N] token -> forward row, or -1 (not computed)
  int *count;         // device scalar: forward rows
  float *kappa;       // [N] per forward row
  uint8_t *flag;      // [N] per forward row
  size_t bytes;       // total size of the cache buffer
};
LogprobCache logprob_cache_view(void *base, int64_t N, int32_t V);

size_t tc_ws_bytes(int64_t N, int32_t h, int32_t V);
sao_status tc_fwd(const void *H, const void *W, const int32_t *y, const uint8_t *row_mask, int64_t N,
                  int32_t h, int32_t V, float *logp, float *lse, unsigned int *err, void *ws, size_t ws_bytes,
                  const LogprobCache *cache, cudaStream_t s);
sao_status tc_bwd(const void *H, const void *W, const int32_t *y, const float *lse, const float *G,
                  int64_t N, int32_t h, int32_t V, void *dH, float *dW, int accumulate, unsigned int *err,
                  void *ws, size_t ws_bytes, const LogprobCache *cache, cudaStream_t s);

}  // namespace sao
