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

// Largest b in [0, B-1] with cu[b] <= t (the trajectory holding token t).
__device__ __forceinline__ int find_traj(const int32_t *cu, int B, int64_t t) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (int64_t(__ldg(cu + mid)) <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

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

// First trajectory of every warp chunk (one binary search per chunk).
__global__ void chunk_first_kernel(const int32_t *cu, int B, int64_t N, int nchunks, int *chunk_first) {
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= nchunks) return;
  const int64_t t = int64_t(q) * kSegChunk;
  chunk_first[q] = find_traj(cu, B, t < N ? t : N - 1);
}

// Number of action tokens per trajectory; nact must start at zero. One warp
// per chunk, 8 warps per CTA; in each 512-token window of the chunk lane l
// reads tokens 16l .. 16l+15 (one contiguous 512-byte warp load), and each
// lane's trajectory walk only moves forward.
__global__ void __launch_bounds__(256) action_count_kernel(const uint8_t *m, const int32_t *cu_g, int B, int64_t N,
                                                           int nchunks, const int *chunk_first, int *nact) {
  __shared__ int32_t s_cu_all[8][kCuCap];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q = blockIdx.x * 8 + warp;
  if (q >= nchunks) return;
  int blo, bhi;
  const CuView cu = stage_chunk(cu_g, B, nchunks, chunk_first, q, lane, s_cu_all[warp], blo, bhi);
  const int64_t c0 = int64_t(q) * kSegChunk;
  int b = blo;
  int64_t next_end = cu[b + 1];
  int cnt = 0;
  const bool aligned = (reinterpret_cast<uintptr_t>(m) & 15u) == 0;
#pragma unroll 1
  for (int g = 0; g < kSegChunk / 512; ++g) {
    const int64_t t0 = c0 + int64_t(g) * 512 + int64_t(lane) * 16;
    if (t0 >= N) break;
    uint32_t w[4] = {0u, 0u, 0u, 0u};
    if (aligned && t0 + 16 <= N) {
      const uint4 x = __ldg(reinterpret_cast<const uint4 *>(m + t0));
      w[0] = x.x;
      w[1] = x.y;
      w[2] = x.z;
      w[3] = x.w;
    } else {
      for (int k = 0; k < 16; ++k) {
        const int64_t t = t0 + k;
        if (t < N && m[t] != 0) w[k >> 2] |= 1u << (8 * (k & 3));
      }
    }
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int64_t t = t0 + k;
      if (t >= N) break;
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
      cnt += ((w[k >> 2] >> (8 * (k & 3))) & 0xffu) != 0u;
    }
  }
  const unsigned peers = __match_any_sync(0xffffffffu, b);
  const int tot = __reduce_add_sync(peers, cnt);
  if (lane == __ffs(peers) - 1 && tot) atomicAdd(nact + b, tot);
}

}  // namespace

}  // namespace seg
}  // namespace sao
