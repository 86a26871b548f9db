// Step-level GAE (App. A.1): the advantage is computed per step (one
// conversation turn = a maximal run of action tokens inside a trajectory) and
// broadcast to the step's tokens.
//
//   1. flag trajectory starts, then step starts (an action token that opens a
//      trajectory or follows a non-action token), and compact the step starts
//      into an ordered step list (count on the device);
//   2. one warp per step finds the step's end and reduces its token values
//      (fp64 sum for the step average, or the last value);
//   3. one thread per trajectory runs the backward GAE over its steps in fp64
//      (steps are few, so fp64 costs nothing here), with the length-adaptive
//      lambda counted in steps;
//   4. one warp per step writes the step's advantage, value target and
//      value-loss mask to its tokens (everything else was zeroed).
#include <stdint.h>

#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {
namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerBlock = 4096;

__global__ void mark_traj_starts(const int32_t *cu, int B, int64_t N, uint8_t *traj_start) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int64_t t = cu[b];
  if (t >= 0 && t < N && cu[b + 1] > t) traj_start[t] = 1;
}

__device__ __forceinline__ bool step_start(const uint8_t *m, const uint8_t *traj_start, int64_t t) {
  return m[t] != 0 && (t == 0 || traj_start[t] != 0 || m[t - 1] == 0);
}

__global__ void __launch_bounds__(kThreads) step_count_kernel(const uint8_t *m, const uint8_t *ts, int64_t N,
                                                              int *block_count) {
  const int64_t r0 = int64_t(blockIdx.x) * kRowsPerBlock;
  int c = 0;
  for (int i = threadIdx.x; i < kRowsPerBlock; i += kThreads) {
    const int64_t t = r0 + i;
    if (t < N) c += step_start(m, ts, t);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __shared__ int sh[kThreads / 32];
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < kThreads / 32; ++w) s += sh[w];
    block_count[blockIdx.x] = s;
  }
}

__global__ void __launch_bounds__(1024) step_scan_kernel(int *block_count, int nblocks, int *total) {
  __shared__ int sh[1024];
  const int per = (nblocks + 1023) / 1024;
  const int b0 = threadIdx.x * per;
  int s = 0;
  for (int i = 0; i < per; ++i)
    if (b0 + i < nblocks) s += block_count[b0 + i];
  sh[threadIdx.x] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const int v = threadIdx.x >= o ? sh[threadIdx.x - o] : 0;
    __syncthreads();
    sh[threadIdx.x] += v;
    __syncthreads();
  }
  int run = threadIdx.x ? sh[threadIdx.x - 1] : 0;
  for (int i = 0; i < per; ++i)
    if (b0 + i < nblocks) {
      const int c = block_count[b0 + i];
      block_count[b0 + i] = run;
      run += c;
    }
  if (threadIdx.x == 1023) *total = sh[1023];
}

__global__ void __launch_bounds__(kThreads) step_scatter_kernel(const uint8_t *m, const uint8_t *ts, int64_t N,
                                                                const int *block_offset, int *step_first) {
  const int64_t r0 = int64_t(blockIdx.x) * kRowsPerBlock;
  __shared__ int sh[kThreads / 32];
  __shared__ int base;
  if (threadIdx.x == 0) base = block_offset[blockIdx.x];
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i0 = 0; i0 < kRowsPerBlock; i0 += kThreads) {
    const int64_t t = r0 + i0 + threadIdx.x;
    const bool a = t < N && step_start(m, ts, t);
    const unsigned bal = __ballot_sync(0xffffffffu, a);
    if (lane == 0) sh[warp] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int w = 0; w < kThreads / 32; ++w) {
      before += (w < warp) ? sh[w] : 0;
      total += sh[w];
    }
    if (a) step_first[base + before + __popc(bal & ((1u << lane) - 1u))] = int(t);
    __syncthreads();
    if (threadIdx.x == 0) base += total;
    __syncthreads();
  }
}

__device__ __forceinline__ int traj_of(const int32_t *cu, int B, int64_t t) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (int64_t(cu[mid]) <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

struct StepInfo {
  double v;    // step value V(S)
  int end;     // one past the step's last token
  int traj;    // trajectory of the step
};

// One warp per step: end of the run of action tokens and the step value.
__global__ void __launch_bounds__(kThreads) step_reduce_kernel(const float *values, const uint8_t *m,
                                                               const uint8_t *ts, const int32_t *cu, int B,
                                                               int64_t N, const int *step_first,
                                                               const int *nsteps, int mode, StepInfo *info) {
  const int lane = threadIdx.x & 31;
  const int S = *nsteps;
  for (int s = (blockIdx.x * kThreads + threadIdx.x) >> 5; s < S; s += (gridDim.x * kThreads) >> 5) {
    const int64_t first = step_first[s];
    double sum = 0.0;
    int64_t end = -1;
    for (int64_t t0 = first;; t0 += 32) {
      const int64_t t = t0 + lane;
      const bool in = t < N && m[t] != 0 && (t == first || ts[t] == 0);
      const unsigned bal = __ballot_sync(0xffffffffu, in);
      const unsigned run = ~bal ? (__ffs(~bal) - 1) : 32;  // tokens of this step in the 32-window
      if (lane < int(run)) sum += double(values[t]);
      if (run < 32) {
        end = t0 + run;
        break;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) {
      StepInfo si;
      si.end = int(end);
      si.v = mode == SAO_STEP_LAST ? double(values[end - 1]) : sum / double(end - first);
      si.traj = traj_of(cu, B, first);
      info[s] = si;
    }
  }
}

// One thread per trajectory: backward GAE over its steps, in fp64.
__global__ void step_gae_kernel(const float *rewards, const int32_t *cu, int B, const int *step_first,
                                const int *nsteps, StepInfo *info, float gamma, float lam, float lam_c,
                                float alpha, float2 *out /*[S] (adv, ret)*/) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int S = *nsteps;
  // steps of trajectory b: first steps whose first token lies in [cu[b], cu[b+1])
  auto lower = [&](int64_t t) {
    int lo = 0, hi = S;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (int64_t(step_first[mid]) < t) lo = mid + 1;
      else hi = mid;
    }
    return lo;
  };
  const int s0 = lower(cu[b]), s1 = lower(cu[b + 1]);
  const int n = s1 - s0;
  if (n <= 0) return;
  double lb = lam;
  if (alpha > 0.f) {
    lb = 1.0 - 1.0 / (double(alpha) * double(n));
    lb = lb < 0.0 ? 0.0 : (lb > 1.0 ? 1.0 : lb);
  }
  const double g = gamma, ap = g * lb, ac = g * double(lam_c);
  double Ap = 0.0, Ac = 0.0, v_next = 0.0;
  double r = rewards[b];
  for (int s = s1 - 1; s >= s0; --s) {
    const double v = info[s].v;
    const double delta = r + g * v_next - v;
    Ap = delta + ap * Ap;
    Ac = delta + ac * Ac;
    out[s] = make_float2(float(Ap), float(Ac + v));
    v_next = v;
    r = 0.0;
  }
}

// One warp per step: broadcast to the step's tokens.
__global__ void __launch_bounds__(kThreads) step_broadcast_kernel(const int *step_first, const int *nsteps,
                                                                  const StepInfo *info, const float2 *out,
                                                                  int mode, float *adv, float *ret,
                                                                  uint8_t *vmask) {
  const int lane = threadIdx.x & 31;
  const int S = *nsteps;
  for (int s = (blockIdx.x * kThreads + threadIdx.x) >> 5; s < S; s += (gridDim.x * kThreads) >> 5) {
    const int first = step_first[s], end = info[s].end;
    const float2 o = out[s];
    for (int t = first + lane; t < end; t += 32) {
      adv[t] = o.x;
      ret[t] = o.y;
      if (vmask) vmask[t] = (mode == SAO_STEP_AVERAGE || t == end - 1) ? 1 : 0;
    }
  }
}

}  // namespace

size_t step_gae_ws_bytes(int64_t N, int64_t B) {
  (void)B;
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  return round256(size_t(N)) + round256(sizeof(int) * (nblocks + 1)) + round256(sizeof(int) * 4) +
         round256(sizeof(int) * N) + round256(sizeof(StepInfo) * N) + round256(sizeof(float2) * N);
}

sao_status step_gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu, int32_t B,
                           int64_t N, float gamma, float lam, float lam_c, float alpha, int mode, float *adv,
                           float *ret, uint8_t *vmask, void *ws_body, size_t body_bytes, cudaStream_t s) {
  if (N == 0) return SAO_OK;
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  Carver c(ws_body, body_bytes);
  uint8_t *ts = c.take<uint8_t>(size_t(N));
  int *block = c.take<int>(size_t(nblocks) + 1);
  int *nsteps = c.take<int>(4);
  int *step_first = c.take<int>(size_t(N));
  StepInfo *info = c.take<StepInfo>(size_t(N));
  float2 *out = c.take<float2>(size_t(N));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the step-level advantages");
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  SAO_CUDA_TRY(cudaMemsetAsync(ts, 0, size_t(N), s));
  SAO_CUDA_TRY(cudaMemsetAsync(adv, 0, sizeof(float) * size_t(N), s));
  SAO_CUDA_TRY(cudaMemsetAsync(ret, 0, sizeof(float) * size_t(N), s));
  if (vmask) SAO_CUDA_TRY(cudaMemsetAsync(vmask, 0, size_t(N), s));
  int slot = launch_begin("step_gae_segments", s);
  mark_traj_starts<<<unsigned((B + 255) / 256), 256, 0, s>>>(cu, B, N, ts);
  step_count_kernel<<<unsigned(nblocks), kThreads, 0, s>>>(m, ts, N, block);
  step_scan_kernel<<<1, 1024, 0, s>>>(block, int(nblocks), nsteps);
  step_scatter_kernel<<<unsigned(nblocks), kThreads, 0, s>>>(m, ts, N, block, step_first);
  SAO_TRY(launch_end(slot, s));
  const unsigned warps_grid = unsigned(di.sm_count * 8);
  slot = launch_begin("step_gae_reduce", s);
  step_reduce_kernel<<<warps_grid, kThreads, 0, s>>>(values, m, ts, cu, B, N, step_first, nsteps, mode, info);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("step_gae_scan", s);
  step_gae_kernel<<<unsigned((B + 127) / 128), 128, 0, s>>>(rewards, cu, B, step_first, nsteps, info, gamma, lam,
                                                           lam_c, alpha, out);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("step_gae_broadcast", s);
  step_broadcast_kernel<<<warps_grid, kThreads, 0, s>>>(step_first, nsteps, info, out, mode, adv, ret, vmask);
  return launch_end(slot, s);
}

}  // namespace sao
