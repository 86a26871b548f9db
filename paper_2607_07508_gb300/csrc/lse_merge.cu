// Merge of the vocabulary-tile softmax partials into lse and logp (Eq. 1-2).
#include <math.h>

#include "logprobs_common.cuh"
#include "sao_common.cuh"

namespace sao {
namespace {

__global__ void __launch_bounds__(256) lse_merge_kernel(const float2 *__restrict__ part, int nvt,
                                                        const float *__restrict__ zy, const int32_t *__restrict__ y,
                                                        const uint8_t *__restrict__ row_mask,
                                                        const int *__restrict__ pos, int64_t N, int V,
                                                        float *logp, float *lse, unsigned int *err) {
  const int64_t row = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (row >= N) return;
  if (row_mask != nullptr && row_mask[row] == 0) {
    logp[row] = 0.f;
    lse[row] = 0.f;
    return;
  }
  // partials of a compacted forward are stored at the row's compact index
  int64_t src = row;
  if (pos != nullptr) {
    const int i = pos[row];
    if (i < 0) {
      logp[row] = 0.f;
      lse[row] = 0.f;
      return;
    }
    src = i;
  }
  // one online pass: (m, s) = running maximum and sum of exp(z - m); four
  // tiles' partials in flight per thread
  float m = -INFINITY, s = 0.f;
  auto merge = [&](float2 p) {
    const float mn = fmaxf(m, p.x);
    s = fmaf(s, expf(m - mn), p.y * expf(p.x - mn));  // every tile holds a finite maximum
    m = mn;
  };
  int j = 0;
  for (; j + 4 <= nvt; j += 4) {
    float2 p[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) p[u] = __ldcs(part + int64_t(j + u) * N + src);
#pragma unroll
    for (int u = 0; u < 4; ++u) merge(p[u]);
  }
  for (; j < nvt; ++j) merge(__ldcs(part + int64_t(j) * N + src));
  const float l = m + logf(s);
  lse[row] = l;
  const int yy = y[row];
  if (yy >= 0 && yy < V) {
    logp[row] = zy[src] - l;
  } else {
    logp[row] = __int_as_float(0x7fc00000);
    raise_device_error(err, SAO_DEVERR_TOKEN_ID);
  }
}

}  // namespace

sao_status lse_merge_launch(const float2 *part, int nvt, const float *zy, const int32_t *y,
                            const uint8_t *row_mask, const int *pos, int64_t N, int32_t V, float *logp, float *lse,
                            unsigned int *err, cudaStream_t s) {
  const int64_t grid = (N + 255) / 256;
  int slot = launch_begin("lse_merge", s);
  lse_merge_kernel<<<unsigned(grid), 256, 0, s>>>(part, nvt, zy, y, row_mask, pos, N, V, logp, lse, err);
  return launch_end(slot, s);
}

}  // namespace sao
