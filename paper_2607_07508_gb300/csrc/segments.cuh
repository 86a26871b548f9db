// Helpers for kernels that walk packed trajectories (cu_seqlens) in warp
// chunks of kSegChunk tokens: the trajectory of each chunk's first token, a
// view of a chunk's cu_seqlens slice staged in shared memory, and the number
// of action tokens per trajectory.
#pragma once

#include <stdint.h>

namespace sao {
namespace seg {

constexpr int kItems = 32;               // tokens per lane (one bit each in a uint32)
constexpr int kSegChunk = 32 * kItems;   // tokens per warp chunk
constexpr int kCuCap = 128;              // cu_seqlens entries staged per warp
constexpr int kCountChunks = 8;          // chunks per warp in action_count_kernel
constexpr int kCastChunks = 2;           // chunks per warp in traj_broadcast_kernel

// CTAs (of 8 warps) of action_count_kernel for nchunks chunks.
__host__ __device__ constexpr unsigned action_count_grid(int nchunks) {
  return unsigned((nchunks + 8 * kCountChunks - 1) / (8 * kCountChunks));
}
// CTAs (of 8 warps) of traj_broadcast_kernel for nchunks chunks.
__host__ __device__ constexpr unsigned broadcast_grid(int nchunks) {
  return unsigned((nchunks + 8 * kCastChunks - 1) / (8 * kCastChunks));
}

// cu_seqlens entries [blo, blo + n) of one chunk, read from shared memory
// when the slice fits there, else from global memory.
struct CuView {
  const int32_t *g;
  const int32_t *s;
  int blo;
  bool in_smem;
  __device__ __forceinline__ int64_t operator[](int b) const { return in_smem ? s[b - blo] : __ldg(g + b); }
  // largest b in [lo, hi] with cu[b] <= t
  __device__ __forceinline__ int find(int lo, int hi, int64_t t) const {
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if ((*this)[mid] <= t) lo = mid;
      else hi = mid - 1;
    }
    return lo;
  }
};

// Stages the cu_seqlens slice of warp chunk q into `s_cu` (kCuCap entries) and
// returns the view; blo/bhi are the first/last trajectories the chunk can touch.
__device__ __forceinline__ CuView stage_chunk(const int32_t *cu, int B, int nchunks, const int *chunk_first, int q,
                                              int lane, int32_t *s_cu, int &blo, int &bhi) {
  blo = __ldg(chunk_first + q);
  bhi = q + 1 < nchunks ? __ldg(chunk_first + q + 1) : B - 1;
  const int ncu = bhi - blo + 2;  // cu[blo .. bhi + 1]
  const CuView v{cu, s_cu, blo, ncu <= kCuCap};
  if (v.in_smem)
    for (int i = lane; i < ncu; i += 32) s_cu[i] = __ldg(cu + blo + i);
  __syncwarp();
  return v;
}

// The kernels below get internal linkage: each translation unit that
// includes this header launches its own copy.
namespace {

// First trajectory of every warp chunk, by trajectory: chunk q gets b when
// its first token lies in b (cu[b] <= q * kSegChunk < cu[b + 1]), so with a
// valid cu_seqlens every chunk is written once, by the one trajectory holding
// its first token (empty trajectories write none). chunk_first must start
// zeroed: a malformed cu_seqlens then still leaves every entry a trajectory
// index, so the passes that read it stay inside cu_seqlens.
// `first`, `step`: the entries one thread writes (0, 1 alone; lane, 32 for a
// warp sharing one trajectory).
__device__ __forceinline__ void chunk_first_of(const int32_t *cu, int b, int64_t N, int nchunks, int *chunk_first,
                                               int first = 0, int step = 1) {
  int64_t t0 = cu[b], t1 = cu[b + 1];
  t0 = t0 < 0 ? 0 : (t0 > N ? N : t0);
  t1 = t1 < 0 ? 0 : (t1 > N ? N : t1);
  const int64_t q0 = (t0 + kSegChunk - 1) / kSegChunk, q1 = (t1 + kSegChunk - 1) / kSegChunk;
#pragma unroll 1
  for (int64_t q = q0 + first; q < q1 && q < nchunks; q += step) chunk_first[q] = b;
}
// One thread per trajectory. Grid: (B + 255) / 256 CTAs of 256 threads.
__global__ void __launch_bounds__(256) chunk_first_kernel(const int32_t *cu, int B, int64_t N, int nchunks,
                                                          int *chunk_first) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B) chunk_first_of(cu, b, N, nchunks, chunk_first);
}
__host__ __device__ constexpr unsigned chunk_first_grid(int B) { return unsigned((B + 255) / 256); }

// Number of action tokens per trajectory; nact must start at zero. One warp
// per kCountChunks consecutive chunks, 8 warps per CTA (grid:
// action_count_grid). A lane's 4 tokens inside its current trajectory are
// counted with one byte-wise popcount; only groups that cross a trajectory
// end take the per-token walk. Each lane adds its count to a trajectory's
// total when it leaves it, and the lanes that end in the same trajectory add
// theirs together.
__global__ void __launch_bounds__(256) action_count_kernel(const uint8_t *m, const int32_t *cu_g, int B, int64_t N,
                                                           int nchunks, const int *chunk_first, int *nact) {
  __shared__ int32_t s_cu_all[8][kCuCap];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q0 = (blockIdx.x * 8 + warp) * kCountChunks;
  if (q0 >= nchunks) return;
  const int q1 = q0 + kCountChunks < nchunks ? q0 + kCountChunks : nchunks;
  const int blo = __ldg(chunk_first + q0);
  const int bhi = q1 < nchunks ? __ldg(chunk_first + q1) : B - 1;
  const int ncu = bhi - blo + 2;  // cu[blo .. bhi + 1]
  const CuView cu{cu_g, s_cu_all[warp], blo, ncu <= kCuCap};
  if (cu.in_smem)
    for (int i = lane; i < ncu; i += 32) s_cu_all[warp][i] = __ldg(cu_g + blo + i);
  __syncwarp();
  const int64_t c0 = int64_t(q0) * kSegChunk;
  const int64_t c1 = int64_t(q1) * kSegChunk < N ? int64_t(q1) * kSegChunk : N;
  int b = blo;
  int64_t next_end = cu[b + 1];
  int cnt = 0;
  const bool aligned = (reinterpret_cast<uintptr_t>(m) & 3u) == 0;
  // 128-token groups, lane l taking tokens 4l .. 4l+3 (each warp load reads 128
  // contiguous bytes); the mask words of 8 groups are loaded together, so a
  // warp waits for one load latency per 1024 tokens; a lane's tokens only
  // increase, so its walk only moves forward
#pragma unroll 1
  for (int64_t base = c0; base < c1; base += 8 * 128) {
    uint32_t u[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t t0 = base + j * 128 + int64_t(lane) * 4;
      u[j] = (aligned && t0 + 4 <= c1) ? __ldg(reinterpret_cast<const uint32_t *>(m + t0)) : 0u;
    }
    if (aligned && base + 8 * 128 <= c1 && base + 8 * 128 <= next_end) {
      // the whole window inside the lane's current trajectory (the common case)
#pragma unroll
      for (int j = 0; j < 8; ++j) cnt += __popc(((u[j] & 0x7f7f7f7fu) + 0x7f7f7f7fu | u[j]) & 0x80808080u);
      continue;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t t0 = base + j * 128 + int64_t(lane) * 4;
      if (t0 >= c1) break;
      if (aligned && t0 + 4 <= c1 && t0 + 4 <= next_end) {  // all 4 tokens in trajectory b
        cnt += __popc(((u[j] & 0x7f7f7f7fu) + 0x7f7f7f7fu | u[j]) & 0x80808080u);
        continue;
      }
      for (int k = 0; k < 4; ++k) {
        const int64_t t = t0 + k;
        if (t >= c1) break;
        if (t >= next_end) {
          const int nb0 = b;
          while (b < bhi && t >= next_end) {
            ++b;
            next_end = cu[b + 1];
          }
          if (b != nb0 && cnt) {
            atomicAdd(nact + nb0, cnt);
            cnt = 0;
          }
        }
        cnt += m[t] != 0;
      }
    }
  }
  const unsigned peers = __match_any_sync(0xffffffffu, b);
  const int tot = __reduce_add_sync(peers, cnt);
  if (lane == __ffs(peers) - 1 && tot) atomicAdd(nact + b, tot);
}

// adv[t] = a_traj[b] on the action tokens of trajectory b, 0 on every other
// token; every token below N is written (cu_seqlens covers [0, N)). Grid:
// broadcast_grid, kCastChunks chunks per warp (its stores run in one short
// wave per chunk pair, so small units keep the SMs busy to the end); in 128-token
// groups lane l takes 4 tokens (a 4-byte mask load, a float4 store); a group
// inside the lane's current trajectory takes no per-token work.
// kValues: also ret[t] = a_traj[b] and adv[t] = a_traj[b] - values[t] on the
// action tokens (0 elsewhere): the GAE of a trajectory whose recursion
// telescopes (gamma = lambda = 1: the advantage is its reward minus the
// value, the return its reward), with the values read by float4 as well.
template <bool kValues>
__global__ void __launch_bounds__(256) traj_broadcast_kernel(const float *a_traj, const uint8_t *m,
                                                             const int32_t *cu_g, int B, int64_t N, int nchunks,
                                                             const int *chunk_first, float *adv,
                                                             const float *values, float *ret) {
  __shared__ int32_t s_cu_all[8][kCuCap];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q0 = (blockIdx.x * 8 + warp) * kCastChunks;
  if (q0 >= nchunks) return;
  const int q1 = q0 + kCastChunks < nchunks ? q0 + kCastChunks : nchunks;
  const int blo = __ldg(chunk_first + q0);
  const int bhi = q1 < nchunks ? __ldg(chunk_first + q1) : B - 1;
  const int ncu = bhi - blo + 2;  // cu[blo .. bhi + 1]
  const CuView cu{cu_g, s_cu_all[warp], blo, ncu <= kCuCap};
  if (cu.in_smem)
    for (int i = lane; i < ncu; i += 32) s_cu_all[warp][i] = __ldg(cu_g + blo + i);
  __syncwarp();
  const int64_t c0 = int64_t(q0) * kSegChunk;
  const int64_t c1 = int64_t(q1) * kSegChunk < N ? int64_t(q1) * kSegChunk : N;
  int b = blo;
  int64_t next_end = cu[b + 1];
  float v = __ldg(a_traj + b);
  uintptr_t al = reinterpret_cast<uintptr_t>(m) | reinterpret_cast<uintptr_t>(adv);
  if (kValues) al |= reinterpret_cast<uintptr_t>(values) | reinterpret_cast<uintptr_t>(ret);
  const bool aligned = (al & 15u) == 0;
  // 128-token groups: lane l takes tokens 4l .. 4l+3, so each warp load reads
  // 128 contiguous bytes and each warp store writes 512; the mask words of 8
  // groups are loaded together, so a warp waits for one load latency per
  // 1024 tokens instead of one per group
#pragma unroll 1
  for (int64_t base = c0; base < c1; base += 8 * 128) {
    uint32_t u[8];
    float4 x[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t t0 = base + j * 128 + int64_t(lane) * 4;
      const bool full = aligned && t0 + 4 <= c1;
      u[j] = full ? __ldg(reinterpret_cast<const uint32_t *>(m + t0)) : 0u;
      if (kValues) x[j] = full ? __ldcs(reinterpret_cast<const float4 *>(values + t0)) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t t0 = base + j * 128 + int64_t(lane) * 4;
      if (t0 >= c1) break;
      if (aligned && t0 + 4 <= c1 && t0 + 4 <= next_end) {  // all 4 tokens in trajectory b
        const uint32_t w = u[j];
        const bool a0 = (w & 0xffu) != 0u, a1 = (w & 0xff00u) != 0u, a2 = (w & 0xff0000u) != 0u,
                   a3 = (w & 0xff000000u) != 0u;
        if (kValues) {
          __stcs(reinterpret_cast<float4 *>(adv + t0),
                 make_float4(a0 ? __fsub_rn(v, x[j].x) : 0.f, a1 ? __fsub_rn(v, x[j].y) : 0.f,
                             a2 ? __fsub_rn(v, x[j].z) : 0.f, a3 ? __fsub_rn(v, x[j].w) : 0.f));
          __stcs(reinterpret_cast<float4 *>(ret + t0), make_float4(a0 ? v : 0.f, a1 ? v : 0.f, a2 ? v : 0.f,
                                                                   a3 ? v : 0.f));
        } else {
          __stcs(reinterpret_cast<float4 *>(adv + t0), make_float4(a0 ? v : 0.f, a1 ? v : 0.f, a2 ? v : 0.f,
                                                                   a3 ? v : 0.f));
        }
        continue;
      }
      for (int k = 0; k < 4; ++k) {
        const int64_t t = t0 + k;
        if (t >= c1) break;
        if (t >= next_end) {
          while (b < bhi && t >= next_end) {
            ++b;
            next_end = cu[b + 1];
          }
          v = __ldg(a_traj + b);
        }
        const bool act = m[t] != 0;
        if (kValues) {
          adv[t] = act ? __fsub_rn(v, values[t]) : 0.f;
          ret[t] = act ? v : 0.f;
        } else {
          adv[t] = act ? v : 0.f;
        }
      }
    }
  }
}

}  // namespace

}  // namespace seg
}  // namespace sao
