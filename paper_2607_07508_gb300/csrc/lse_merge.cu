// Merge of the vocabulary-tile softmax partials into lse and logp (Eq. 1-2).
#include <math.h>

#include "logprobs_common.cuh"
#include "sao_common.cuh"

namespace sao {
namespace {

// Eight threads per row (four rows per warp): thread k of a row merges tiles
// k, k + 8, ... in one online pass with four loads in flight, then the eight
// (max, sum) pairs are combined by a fixed shuffle tree. Each warp load is
// four consecutive rows of eight tiles: eight full 32-byte sectors.
constexpr int kSub = 8;

__global__ void __launch_bounds__(256) lse_merge_kernel(const float2 *__restrict__ part, int nvt,
                                                        const float *__restrict__ zy, const int32_t *__restrict__ y,
                                                        const uint8_t *__restrict__ row_mask,
                                                        const int *__restrict__ pos, int64_t N, int V,
                                                        float *logp, float *lse, unsigned int *err) {
  const int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t row = t / kSub;
  const int sub = int(t % kSub);
  // a row's 8 threads are 8 consecutive lanes of one warp; rows past N only join the shuffles
  const bool live = row < N;
  bool skip = !live || (row_mask != nullptr && row_mask[row] == 0);
  // partials of a compacted forward are stored at the row's compact index
  int64_t src = row;
  if (!skip && pos != nullptr) {
    const int i = pos[row];
    if (i < 0)
      skip = true;
    else
      src = i;
  }
  // (m, s) = running maximum and sum of exp(z - m)
  float m = -INFINITY, s = 0.f;
  auto merge = [&](float pm, float ps) {
    const float mn = fmaxf(m, pm);
    if (mn == -INFINITY) return;  // nothing merged on either side yet
    s = fmaf(s, expf(m - mn), ps * expf(pm - mn));
    m = mn;
  };
  if (!skip) {
    int j = sub;
    for (; j + 3 * kSub < nvt; j += 4 * kSub) {
      float2 p[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) p[u] = __ldcs(part + int64_t(j + u * kSub) * N + src);
#pragma unroll
      for (int u = 0; u < 4; ++u) merge(p[u].x, p[u].y);
    }
    for (; j < nvt; j += kSub) {
      const float2 p = __ldcs(part + int64_t(j) * N + src);
      merge(p.x, p.y);
    }
  }
#pragma unroll
  for (int o = 1; o < kSub; o <<= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m, o), os = __shfl_xor_sync(0xffffffffu, s, o);
    merge(om, os);
  }
  if (!live || sub != 0) return;
  if (skip) {
    logp[row] = 0.f;
    lse[row] = 0.f;
    return;
  }
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
  const int64_t grid = (N * kSub + 255) / 256;
  int slot = launch_begin("lse_merge", s);
  lse_merge_kernel<<<unsigned(grid), 256, 0, s>>>(part, nvt, zy, y, row_mask, pos, N, V, logp, lse, err);
  return launch_end(slot, s);
}

}  // namespace sao
