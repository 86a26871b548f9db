// The paper's comparison arms (§4.2): the clipped surrogate of the
// Preliminaries' unified objective with asymmetric ("clip-higher") bounds and
// token or per-sequence normalisation, and GRPO's group-normalised advantage.
//
// The surrogate walks the packed trajectories in 1024-token warp chunks (like
// the advantage scan) so every token knows its trajectory's action count for
// the per-sequence weight; per-warp partial sums are added in a fixed order by
// a one-CTA finaliser, so results are deterministic.
#include <math.h>
#include <stdint.h>

#include "sao_common.cuh"
#include "sao_internal.h"
#include "dfloat.cuh"
#include "segments.cuh"

namespace sao {
namespace {

using seg::CuView;
using seg::kCuCap;
using seg::kSegChunk;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// Compensated fp32 sum (Knuth two-sum): about 48 bits without the fp64 pipe.
struct Sum2 {
  float hi = 0.f, lo = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float s = __fadd_rn(hi, x);
    const float bb = __fsub_rn(s, hi);
    lo = __fadd_rn(lo, __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(x, bb)));
    hi = s;
  }
  __device__ __forceinline__ void merge(float ohi, float olo) {
    add(ohi);
    lo = __fadd_rn(lo, olo);
  }
  __device__ __forceinline__ double value() const { return double(hi) + double(lo); }
};

struct Norms {
  long long n_action;  // action tokens
  long long n_seq;     // trajectories with at least one action token
};

// Sums the per-trajectory action counts: one CTA of 1024 threads, thread i
// taking entries i, i + 1024, ... with eight loads in flight (integer sums,
// so the order does not matter).
constexpr int kNormThreads = 1024;

__global__ void __launch_bounds__(kNormThreads) norms_kernel(const int *nact, int B, Norms *out) {
  long long n = 0, s = 0;
  constexpr int kU = 8;
  int b = threadIdx.x;
  for (; b + (kU - 1) * kNormThreads < B; b += kU * kNormThreads) {
    int v[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) v[u] = __ldg(nact + b + u * kNormThreads);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      n += v[u];
      s += v[u] > 0;
    }
  }
  for (; b < B; b += kNormThreads) {
    const int v = __ldg(nact + b);
    n += v;
    s += v > 0;
  }
  __shared__ long long sh[2][kNormThreads / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n += __shfl_xor_sync(0xffffffffu, n, o);
    s += __shfl_xor_sync(0xffffffffu, s, o);
  }
  if ((threadIdx.x & 31) == 0) {
    sh[0][threadIdx.x >> 5] = n;
    sh[1][threadIdx.x >> 5] = s;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    Norms r{0, 0};
    for (int w = 0; w < kNormThreads / 32; ++w) {
      r.n_action += sh[0][w];
      r.n_seq += sh[1][w];
    }
    *out = r;
  }
}

struct ClipArgs {
  const float *logp, *old, *adv;
  const uint8_t *m;
  const int32_t *cu;
  int B;
  int64_t N;
  int nchunks;
  const int *chunk_first;
  const int *nact;
  const Norms *norms;
  float lo, hi;
  int seq;             // per-sequence normalisation
  float *coef;         // may be null
  uint8_t *flags;      // may be null
  const float *grad_scale;
  float2 *part_loss;   // [CTAs] compensated (hi, lo)
  int *part_cnt;        // [3][CTAs]
};

// One token of the clipped surrogate: returns the weighted value term and
// writes the coefficient d loss / d logp (before the sign) and the flag. The
// cases are taken by selects in the order not-action, non-finite, clipped
// above, clipped below, kept; a value term is (w * f) * a with f = r, or the
// bound it is clipped to.
__device__ __forceinline__ float clip_token(float lp, float old, float a, bool act, float lo, float hi, float w,
                                            float &coef, uint8_t &flag, int &nl, int &nh, int &nf) {
  const float d = lp - old;
  // zero when d and a are both finite, NaN otherwise
  const bool fin = ((d - d) + (a - a)) == 0.f;
  const float r = expf(d);
  const bool ch = a > 0.f && r > hi;
  const bool cl = a < 0.f && r < lo;
  const float f = ch ? hi : (cl ? lo : r);
  const float t = w * f * a;
  const bool live = act && fin;
  nf += act && !fin;
  nh += live && ch;
  nl += live && cl;
  flag = !act ? uint8_t(SAO_FLAG_NOT_ACTION) : !fin ? uint8_t(SAO_FLAG_NONFINITE) : ch ? uint8_t(2) : cl ? uint8_t(1) : uint8_t(0);
  coef = live && !ch && !cl ? -t : 0.f;
  return live ? t : 0.f;
}

template <bool kBwd>
__global__ void __launch_bounds__(kThreads, 5) clip_loss_kernel(ClipArgs a) {
  __shared__ int32_t s_cu_all[kWarps][kCuCap];
  __shared__ float2 s_sum[kWarps];
  __shared__ int s_cnt[3][kWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q = blockIdx.x * kWarps + warp;
  // a lane's 32 value terms in fp32 (relative error ~1e-6, far inside the 1e-4
  // loss bar); lanes, warps and CTAs are then combined compensated
  float lacc = 0.f;
  int nl = 0, nh = 0, nf = 0;
  if (q < a.nchunks) {
    int blo, bhi;
    const CuView cu = seg::stage_chunk(a.cu, a.B, a.nchunks, a.chunk_first, q, lane, s_cu_all[warp], blo, bhi);
    const Norms nm = *a.norms;
    // fp32 weights (one rounding each, far inside the 1e-5 coefficient bar)
    const float w_tok = nm.n_action > 0 ? __fdiv_rn(1.f, float(nm.n_action)) : 0.f;
    const float inv_seq = nm.n_seq > 0 ? __fdiv_rn(1.f, float(nm.n_seq)) : 0.f;
    const float gscale = kBwd ? __ldg(a.grad_scale) : 1.f;
    // window-major: in each 128-token window of the chunk, lane l takes tokens
    // 4l .. 4l+3, so every warp load and store is one contiguous 512 (or 128)
    // byte access; each lane's trajectory walk still only moves forward
    const int64_t c0 = int64_t(q) * kSegChunk;
    const int64_t N = a.N;
    int b = blo;
    int64_t next_end = cu[b + 1];
    auto weight = [&](int bb) {
      if (!a.seq) return w_tok;
      const int L = __ldg(a.nact + bb);
      return L > 0 ? __fdiv_rn(inv_seq, float(L)) : 0.f;
    };
    float w = weight(b);
    const bool aligned = aligned16_dev(a.logp) && aligned16_dev(a.old) && aligned16_dev(a.adv) &&
                         ((reinterpret_cast<uintptr_t>(a.m) & 3u) == 0) && (a.coef == nullptr || aligned16_dev(a.coef)) &&
                         (a.flags == nullptr || (reinterpret_cast<uintptr_t>(a.flags) & 3u) == 0);
  #pragma unroll 1
    for (int g = 0; g < kSegChunk / 128; ++g) {
      const int64_t tg = c0 + int64_t(g) * 128 + int64_t(lane) * 4;
      const bool vec = aligned && tg + 4 <= N;
      float lp[4], od[4], ad[4];
      bool act[4];
      if (vec) {
        const float4 x = __ldg(reinterpret_cast<const float4 *>(a.logp + tg));
        const float4 y = __ldg(reinterpret_cast<const float4 *>(a.old + tg));
        const float4 z = __ldg(reinterpret_cast<const float4 *>(a.adv + tg));
        const uint32_t mw = __ldg(reinterpret_cast<const unsigned int *>(a.m + tg));
        lp[0] = x.x; lp[1] = x.y; lp[2] = x.z; lp[3] = x.w;
        od[0] = y.x; od[1] = y.y; od[2] = y.z; od[3] = y.w;
        ad[0] = z.x; ad[1] = z.y; ad[2] = z.z; ad[3] = z.w;
#pragma unroll
        for (int i = 0; i < 4; ++i) act[i] = ((mw >> (8 * i)) & 0xffu) != 0u;
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const bool in = tg + i < N;
          lp[i] = in ? a.logp[tg + i] : 0.f;
          od[i] = in ? a.old[tg + i] : 0.f;
          ad[i] = in ? a.adv[tg + i] : 0.f;
          act[i] = in && a.m[tg + i] != 0;
        }
      }
      float cf[4];
      uint8_t fl[4];
      float wt[4] = {w, w, w, w};
      if (a.seq && tg + 3 >= next_end) {
        // the lane's four tokens reach a trajectory end (rare for long trajectories)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int64_t t = tg + i;
          if (t < N && t >= next_end) {
            while (b < bhi && t >= next_end) {
              ++b;
              next_end = cu[b + 1];
            }
            w = weight(b);
          }
          wt[i] = w;
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        lacc += clip_token(lp[i], od[i], ad[i], act[i], a.lo, a.hi, wt[i], cf[i], fl[i], nl, nh, nf);
        if constexpr (kBwd) cf[i] *= gscale;
      }
      if (vec) {
        if (a.coef) *reinterpret_cast<float4 *>(a.coef + tg) = make_float4(cf[0], cf[1], cf[2], cf[3]);
        if (a.flags && !kBwd) *reinterpret_cast<uchar4 *>(a.flags + tg) = make_uchar4(fl[0], fl[1], fl[2], fl[3]);
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (tg + i < N) {
            if (a.coef) a.coef[tg + i] = cf[i];
            if (a.flags && !kBwd) a.flags[tg + i] = fl[i];
          }
      }
    }
  }
  if constexpr (!kBwd) {
    // warp, then CTA (fixed order), in compensated fp32
    Sum2 acc;
    acc.add(lacc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ohi = __shfl_xor_sync(0xffffffffu, acc.hi, o), olo = __shfl_xor_sync(0xffffffffu, acc.lo, o);
      acc.merge(ohi, olo);
      nl += __shfl_xor_sync(0xffffffffu, nl, o);
      nh += __shfl_xor_sync(0xffffffffu, nh, o);
      nf += __shfl_xor_sync(0xffffffffu, nf, o);
    }
    if (lane == 0) {
      s_sum[warp] = make_float2(acc.hi, acc.lo);
      s_cnt[0][warp] = nl;
      s_cnt[1][warp] = nh;
      s_cnt[2][warp] = nf;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      Sum2 t;
      int l = 0, h = 0, f = 0;
      for (int k = 0; k < kWarps; ++k) {
        t.merge(s_sum[k].x, s_sum[k].y);
        l += s_cnt[0][k];
        h += s_cnt[1][k];
        f += s_cnt[2][k];
      }
      a.part_loss[blockIdx.x] = make_float2(t.hi, t.lo);
      a.part_cnt[blockIdx.x] = l;
      a.part_cnt[gridDim.x + blockIdx.x] = h;
      a.part_cnt[2 * gridDim.x + blockIdx.x] = f;
    }
  }
}

// One CTA of 1024 threads sums the per-CTA partials in a fixed order: thread i
// takes partials i, i + 1024, ... (eight loads in flight), then the warps and
// the CTA combine theirs in lane and warp order.
constexpr int kFinThreads = 1024;

__global__ void __launch_bounds__(kFinThreads) clip_finalize_kernel(const float2 *part_loss, const int *part_cnt,
                                                                    int n, const Norms *norms, float *loss,
                                                                    int64_t *counts) {
  Sum2 acc;
  long long l = 0, h = 0, f = 0;
  constexpr int kU = 8;
  int i = threadIdx.x;
  for (; i + (kU - 1) * kFinThreads < n; i += kU * kFinThreads) {
    float2 p[kU];
    int c0[kU], c1[kU], c2[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int j = i + u * kFinThreads;
      p[u] = part_loss[j];
      c0[u] = part_cnt[j];
      c1[u] = part_cnt[n + j];
      c2[u] = part_cnt[2 * n + j];
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      acc.merge(p[u].x, p[u].y);
      l += c0[u];
      h += c1[u];
      f += c2[u];
    }
  }
  for (; i < n; i += kFinThreads) {
    acc.merge(part_loss[i].x, part_loss[i].y);
    l += part_cnt[i];
    h += part_cnt[n + i];
    f += part_cnt[2 * n + i];
  }
  __shared__ float2 sd[kFinThreads / 32];
  __shared__ long long sl[3][kFinThreads / 32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ohi = __shfl_down_sync(0xffffffffu, acc.hi, o), olo = __shfl_down_sync(0xffffffffu, acc.lo, o);
    acc.merge(ohi, olo);
    l += __shfl_down_sync(0xffffffffu, l, o);
    h += __shfl_down_sync(0xffffffffu, h, o);
    f += __shfl_down_sync(0xffffffffu, f, o);
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    sd[w] = make_float2(acc.hi, acc.lo);
    sl[0][w] = l;
    sl[1][w] = h;
    sl[2][w] = f;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    Sum2 T;
    long long L = 0, Hh = 0, F = 0;
    for (int k = 0; k < kFinThreads / 32; ++k) {
      T.merge(sd[k].x, sd[k].y);
      L += sl[0][k];
      Hh += sl[1][k];
      F += sl[2][k];
    }
    *loss = float(-T.value());
    counts[0] = norms->n_action;
    counts[1] = L;
    counts[2] = Hh;
    counts[3] = F;
  }
}

// GRPO: per-trajectory standardised reward within its group. One warp per
// trajectory, 8 per CTA sharing shared-memory tiles of the group ids and
// rewards; lane l takes entries l, l + 32, ... of each tile in batch order
// (compensated fp32), the lanes' partial sums are combined down to lane 0 in
// a fixed order, and the final moments are taken in fp64: the mean, then the
// centred second moment.
constexpr int kTile = 2048;

// Lane 0's total of the 32 lanes' compensated partials (fixed tree order).
__device__ __forceinline__ Sum2 warp_total(Sum2 s) {
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) {
    const float ohi = __shfl_down_sync(0xffffffffu, s.hi, d), olo = __shfl_down_sync(0xffffffffu, s.lo, d);
    s.merge(ohi, olo);
  }
  return s;
}

// flag = 0 when some group id is larger than the next one (the flag starts at
// 1): with non-decreasing ids every group is one contiguous run of the batch.
__global__ void group_sorted_kernel(const int32_t *gid, int B, int *flag) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b + 1 < B && __ldg(gid + b) > __ldg(gid + b + 1)) *flag = 0;
}

// First index of the run of group id g that holds index b (dir = -1), or one
// past its last index (dir = +1), for sorted ids; a warp walks 32 entries per
// step.
__device__ int run_edge(const int32_t *gid, int B, int b, int g, int dir, int lane) {
  int edge = b;
  for (;;) {
    const int i = edge + dir * (1 + lane);
    const bool in = i >= 0 && i < B && __ldg(gid + i) == g;
    const unsigned out = __ballot_sync(0xffffffffu, !in);
    if (out) return edge + dir * (__ffs(out) - 1) + (dir > 0 ? 1 : 0);
    edge += 32 * dir;
  }
}

__global__ void __launch_bounds__(256) group_norm_kernel(const float *R, const int32_t *gid, int B, float eps,
                                                         const int *sorted, float *a_traj, const int32_t *cu,
                                                         int64_t N, int nchunks, int *chunk_first) {
  __shared__ int32_t sg[kTile];
  __shared__ float sr[kTile];
  __shared__ int s_range[2];
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (b < B) seg::chunk_first_of(cu, b, N, nchunks, chunk_first, lane, 32);  // for the broadcast
  const int g = b < B ? gid[b] : 0;
  // The entries to visit: the whole batch, or with non-decreasing ids the runs
  // of this CTA's groups (the same members in the same lane order, so the same
  // sums either way).
  if (threadIdx.x < 32) {
    int lo = 0, hi = B;
    if (*sorted) {
      const int b0 = blockIdx.x * 8, b1 = min(B, b0 + 8) - 1;
      lo = run_edge(gid, B, b0, __ldg(gid + b0), -1, lane);
      hi = run_edge(gid, B, b1, __ldg(gid + b1), +1, lane);
    }
    if (lane == 0) {
      s_range[0] = lo;
      s_range[1] = hi;
    }
  }
  __syncthreads();
  const int lo = s_range[0], hi = s_range[1];
  Sum2 s, s2;
  int n = 0;
  float mu = 0.f;
  // A lane meets its members (entries lane, lane + 32, ...) in batch order;
  // up to 4 of their rewards stay in registers, so when no lane of the CTA has
  // more (groups of tens of trajectories) the second moment needs no second
  // sweep, and it adds the same values in the same order.
  float r0 = 0.f, r1 = 0.f, r2 = 0.f, r3 = 0.f;
  for (int t0 = lo / kTile * kTile; t0 < hi; t0 += kTile) {
    const int klo = max(lo - t0, 0), khi = min(kTile, hi - t0);
    __syncthreads();
    for (int k = klo + int(threadIdx.x); k < khi; k += blockDim.x) {
      sg[k] = gid[t0 + k];
      sr[k] = R[t0 + k];
    }
    __syncthreads();
    if (b >= B) continue;
    for (int k = klo + ((lane - klo) & 31); k < khi; k += 32) {
      if (sg[k] != g) continue;
      const float r = sr[k];
      s.add(r);
      r0 = n == 0 ? r : r0;
      r1 = n == 1 ? r : r1;
      r2 = n == 2 ? r : r2;
      r3 = n == 3 ? r : r3;
      ++n;
    }
  }
  if (b < B) {  // the group's mean, from lane 0 to every lane
    const Sum2 t = warp_total(s);
    const int nt = __reduce_add_sync(0xffffffffu, n);
    mu = __shfl_sync(0xffffffffu, dfl::round(dfl::div_int(dfl::norm(t.hi, t.lo), nt > 0 ? nt : 1)), 0);
  }
  const bool sweep = __syncthreads_or(b < B && n > 4);
  if (!sweep) {
    const float rr[4] = {r0, r1, r2, r3};
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < n) {
        const float d = __fsub_rn(rr[i], mu);
        s2.add(__fmul_rn(d, d));
      }
  } else {
    for (int t0 = lo / kTile * kTile; t0 < hi; t0 += kTile) {
      const int klo = max(lo - t0, 0), khi = min(kTile, hi - t0);
      __syncthreads();
      for (int k = klo + int(threadIdx.x); k < khi; k += blockDim.x) {
        sg[k] = gid[t0 + k];
        sr[k] = R[t0 + k];
      }
      __syncthreads();
      if (b >= B) continue;
      for (int k = klo + ((lane - klo) & 31); k < khi; k += 32) {
        if (sg[k] != g) continue;
        const float d = __fsub_rn(sr[k], mu);
        s2.add(__fmul_rn(d, d));
      }
    }
  }
  if (b >= B) return;
  const Sum2 t = warp_total(s), t2 = warp_total(s2);
  const int nt = __reduce_add_sync(0xffffffffu, n);
  if (lane == 0) {
    // exact mean correction for the rounded mu: var = E[(r - mu)^2] - (mean - mu)^2,
    // in double-float; then (R - mean) rounded once and divided in fp32
    const dfl::F2 mean = dfl::div_int(dfl::norm(t.hi, t.lo), nt);
    const dfl::F2 dm = dfl::sub(mean, dfl::F2{mu, 0.f});
    const dfl::F2 var = dfl::sub(dfl::div_int(dfl::norm(t2.hi, t2.lo), nt), dfl::mul(dm, dm));
    const float v = fmaxf(dfl::round(var), 0.f);
    const float num = dfl::round(dfl::sub(dfl::F2{R[b], 0.f}, mean));
    a_traj[b] = __fdiv_rn(num, __fsqrt_rn(__fadd_rn(v, eps)));
  }
}

// Running-mean baseline. Trajectory b of prompt p sees the window as it stands
// after the k in-batch trajectories of p before it have been recorded: their
// last min(k, window) rewards, plus the slots of the caller's ring buffer that
// those k writes have not overwritten. So every trajectory is independent:
// one warp per trajectory walks the batch backwards from b (most recent
// first, 32 entries per step: a ballot ranks the matches), then the ring
// buffers are updated in a second pass. Sums are compensated fp32 (about 48
// bits), combined in a fixed order; the mean and the advantage in
// double-float.

// In-batch ranks for dense prompt ids (P <= kRankMaxPrompts): counts of each
// prompt per block of kRankBlock trajectories, then their exclusive prefix over
// the blocks (row nblk: each prompt's total), so the rank of b is
// table[b / kRankBlock][p] plus the trajectories of p in b's block before b.
constexpr int kRankBlock = 1024;
constexpr int kRankMaxPrompts = 4096;

__global__ void __launch_bounds__(256) rank_count_kernel(const int32_t *pid, int B, int P, int *table) {
  __shared__ int cnt[kRankMaxPrompts];
  for (int q = threadIdx.x; q < P; q += blockDim.x) cnt[q] = 0;
  __syncthreads();
  const int b0 = blockIdx.x * kRankBlock;
  for (int i = threadIdx.x; i < kRankBlock && b0 + i < B; i += blockDim.x) {
    const int q = pid[b0 + i];
    if (q >= 0 && q < P) atomicAdd(&cnt[q], 1);  // ids outside [0, P) are the caller's error: skipped
  }
  __syncthreads();
  for (int q = threadIdx.x; q < P; q += blockDim.x) table[int64_t(blockIdx.x) * P + q] = cnt[q];
}

// One warp per prompt: exclusive prefix of its per-block counts, 32 blocks at
// a time by a shuffle scan.
__global__ void __launch_bounds__(256) rank_scan_kernel(int *table, int nblk, int P) {
  const int q = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (q >= P) return;
  int run = 0;
  for (int k0 = 0; k0 < nblk; k0 += 32) {
    const int k = k0 + lane;
    const int v = k < nblk ? table[int64_t(k) * P + q] : 0;
    int inc = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, inc, d);
      if (lane >= d) inc += o;
    }
    if (k < nblk) table[int64_t(k) * P + q] = run + inc - v;
    run += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (lane == 0) table[int64_t(nblk) * P + q] = run;
}

// One warp per trajectory b of prompt p: the sum of the rewards of the most
// recent min(k, window) in-batch trajectories of p before b, walking down from
// b - 1 32 entries at a time (lane l takes b - 1 - 32 j - l; a ballot ranks
// the hits, newest first), and k, their number. With the rank table the walk
// stops at the window-th hit and k comes from the table; without it the walk
// runs to the start of the batch. Either way the same hits are summed in the
// same order.
__global__ void __launch_bounds__(256) running_mean_kernel(const float *R, const int32_t *pid, int B, int P,
                                                           const int *table, const float *history,
                                                           const long long *seen, int window, float *a_traj,
                                                           long long *rec, int *rank, const int32_t *cu, int64_t N,
                                                           int nchunks, int *chunk_first) {
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (b >= B) return;
  seg::chunk_first_of(cu, b, N, nchunks, chunk_first, lane, 32);  // for the broadcast
  const int p = pid[b];
  if (p < 0 || p >= P) {  // outside [0, num_prompts): no window to read, advantage 0
    if (lane == 0) {
      a_traj[b] = 0.f;
      rec[b] = -1;
    }
    return;
  }
  Sum2 sum;      // this lane's share, compensated fp32
  int hits = 0;  // warp-uniform
  // four 32-entry slices per step: their ids, then the hit rewards, loaded
  // together; the hits are then taken slice by slice as one slice at a time
  // would (same sums in the same order)
  bool done = false;
  for (int top = b - 1; top >= 0 && !done; top -= 128) {
    int ids[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = top - 32 * u - lane;
      ids[u] = i >= 0 ? __ldg(pid + i) : -1;
    }
    float rw[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) rw[u] = ids[u] == p ? __ldg(R + (top - 32 * u - lane)) : 0.f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (done) break;
      const bool hit = ids[u] == p;
      const unsigned mask = __ballot_sync(0xffffffffu, hit);
      if (hit && hits + __popc(mask & ((1u << lane) - 1u)) < window) sum.add(rw[u]);
      hits += __popc(mask);
      if (table && hits >= window) done = true;
    }
  }
  int k = hits;
  if (table) {  // rank of b: earlier blocks from the table, then b's own block
    const int b0 = b / kRankBlock * kRankBlock;
    k = __ldg(table + int64_t(b / kRankBlock) * P + p);
    for (int i0 = b0; i0 < b; i0 += 128) {
      int ids[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = i0 + 32 * u + lane;
        ids[u] = i < b ? __ldg(pid + i) : -1;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) k += __popc(__ballot_sync(0xffffffffu, ids[u] == p));
    }
  }
  const long long c = seen[p];
  // old slots still holding rewards: the first min(c, window) slots, except the
  // k (cyclic) slots c % window, ..., (c + k - 1) % window written since
  const int valid_old = int(c < window ? c : window);
  if (k < window) {
    const float *h = history + int64_t(p) * window;
    for (int q = lane; q < valid_old; q += 32) {
      const int since = int(((long long)q - c % window + window) % window);  // write order of slot q after c
      if (since >= k) sum.add(h[q]);
    }
  }
  sum = warp_total(sum);
  if (lane == 0) {
    const long long n = (c + k) < window ? (c + k) : window;
    const dfl::F2 mean = n > 0 ? dfl::div_int(dfl::norm(sum.hi, sum.lo), int(n)) : dfl::F2{0.f, 0.f};
    a_traj[b] = dfl::round(dfl::sub(dfl::F2{R[b], 0.f}, mean));
    rec[b] = c + k;  // b's position in its prompt's reward sequence
    if (rank) rank[b] = k;
  }
}

// Records the batch: the last `window` rewards of each prompt go to their ring
// slots (distinct slots), and the prompt's last trajectory advances its count.
// Positions come from the first pass, so this pass never reads `seen`. The
// number of later trajectories of b's prompt is its total minus b's rank when
// the rank table exists; otherwise one warp per trajectory counts them,
// stopping once there are `window` of them.
__global__ void __launch_bounds__(256) running_mean_record_kernel(const float *R, const int32_t *pid, int B, int P,
                                                                  const int *totals, const int *rank,
                                                                  const long long *rec, float *history,
                                                                  long long *seen, int window) {
  __shared__ int32_t sp[kTile];
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int p = b < B ? pid[b] : -1;
  int after = 0;
  if (totals) {
    if (b < B && p >= 0 && p < P) after = totals[p] - 1 - rank[b];
  } else {
    for (int t0 = int(blockIdx.x) * 8 + 1; t0 < B; t0 += kTile) {
      const int len = min(kTile, B - t0);
      __syncthreads();
      for (int i = threadIdx.x; i < len; i += blockDim.x) sp[i] = pid[t0 + i];
      __syncthreads();
      if (b >= B || after >= window) continue;
      for (int i = max(0, b + 1 - t0) + lane; i - lane < len && after < window; i += 32)
        after += __popc(__ballot_sync(0xffffffffu, i < len && sp[i] == p));
    }
  }
  if (b >= B || lane != 0 || rec[b] < 0) return;  // rec < 0: a prompt id outside [0, num_prompts)
  if (after < window) history[int64_t(p) * window + int(rec[b] % window)] = R[b];
  if (after == 0) seen[p] = rec[b] + 1;
}

}  // namespace

size_t baselines_ws_bytes(int64_t N, int64_t B) {
  const int64_t nchunks = (N + kSegChunk - 1) / kSegChunk;
  return round256(sizeof(int) * (nchunks + 1)) + round256(sizeof(int) * (B + 1)) + round256(sizeof(Norms)) +
         round256(sizeof(double) * nchunks) + round256(sizeof(int) * 3 * nchunks) + round256(sizeof(float) * (B + 1)) +
         round256(sizeof(long long) * (B + 1));
}

sao_status clip_loss_launch(const float *logp, const float *old, const float *adv, const uint8_t *m, const int32_t *cu,
                            int32_t B, int64_t N, float eps_low, float eps_high, int norm, float *loss, float *coef,
                            uint8_t *flags, int64_t *counts, const float *grad_loss, void *ws_body,
                            size_t body_bytes, cudaStream_t s) {
  const int64_t nchunks = (N + kSegChunk - 1) / kSegChunk;
  Carver c(ws_body, body_bytes);
  int *chunk_first = c.take<int>(size_t(nchunks) + 1);
  int *nact = c.take<int>(size_t(B) + 1);
  Norms *norms = c.take<Norms>(1);
  float2 *part_loss = c.take<float2>(size_t(nchunks));
  int *part_cnt = c.take<int>(3 * size_t(nchunks));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the clipped surrogate");
  if (N == 0) {
    if (loss) SAO_CUDA_TRY(cudaMemsetAsync(loss, 0, sizeof(float), s));
    if (counts) SAO_CUDA_TRY(cudaMemsetAsync(counts, 0, 4 * sizeof(int64_t), s));
    return SAO_OK;
  }
  // chunk_first and nact start at zero (one memset: nact follows chunk_first)
  SAO_CUDA_TRY(cudaMemsetAsync(chunk_first, 0, size_t(reinterpret_cast<char *>(nact + B) -
                                                       reinterpret_cast<char *>(chunk_first)), s));
  const unsigned grid = unsigned((nchunks + kWarps - 1) / kWarps);
  int slot = launch_begin("clip_loss_counts", s);
  seg::chunk_first_kernel<<<seg::chunk_first_grid(B), 256, 0, s>>>(cu, B, N, int(nchunks), chunk_first);
  seg::action_count_kernel<<<seg::action_count_grid(int(nchunks)), 256, 0, s>>>(m, cu, B, N, int(nchunks),
                                                                                chunk_first, nact);
  norms_kernel<<<1, kNormThreads, 0, s>>>(nact, B, norms);
  SAO_TRY(launch_end(slot, s));
  ClipArgs a;
  a.logp = logp;
  a.old = old;
  a.adv = adv;
  a.m = m;
  a.cu = cu;
  a.B = B;
  a.N = N;
  a.nchunks = int(nchunks);
  a.chunk_first = chunk_first;
  a.nact = nact;
  a.norms = norms;
  a.lo = 1.0f - eps_low;
  a.hi = 1.0f + eps_high;
  a.seq = norm == SAO_NORM_SEQUENCE;
  a.coef = coef;
  a.flags = flags;
  a.grad_scale = grad_loss;
  a.part_loss = part_loss;
  a.part_cnt = part_cnt;
  if (grad_loss) {
    slot = launch_begin("clip_loss_bwd", s);
    clip_loss_kernel<true><<<grid, kThreads, 0, s>>>(a);
    return launch_end(slot, s);
  }
  slot = launch_begin("clip_loss_fwd", s);
  clip_loss_kernel<false><<<grid, kThreads, 0, s>>>(a);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("clip_loss_finalize", s);
  clip_finalize_kernel<<<1, kFinThreads, 0, s>>>(part_loss, part_cnt, int(grid), norms, loss, counts);
  return launch_end(slot, s);
}

// adv[t] = a_traj[trajectory of t] on action tokens, 0 elsewhere, all N tokens
// (chunk_first written by the per-trajectory pass before it).
static sao_status broadcast_launch(const float *a_traj, const uint8_t *m, const int32_t *cu, int32_t B, int64_t N,
                                   const int *chunk_first, float *adv, cudaStream_t s) {
  if (N == 0) return SAO_OK;
  const int64_t nchunks = (N + kSegChunk - 1) / kSegChunk;
  int slot = launch_begin("adv_broadcast", s);
  seg::traj_broadcast_kernel<false><<<seg::broadcast_grid(int(nchunks)), 256, 0, s>>>(
      a_traj, m, cu, B, N, int(nchunks), chunk_first, adv, nullptr, nullptr);
  return launch_end(slot, s);
}

sao_status group_adv_launch(const float *rewards, const int32_t *gid, int32_t B, const uint8_t *m, const int32_t *cu,
                            int64_t N, float eps, float *adv, void *ws_body, size_t body_bytes, cudaStream_t s) {
  Carver c(ws_body, body_bytes);
  float *a_traj = c.take<float>(size_t(B) + 1);
  int *chunk_first = c.take<int>(size_t((N + kSegChunk - 1) / kSegChunk) + 1);
  int *sorted = c.take<int>(1);
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the group advantages");
  if (B == 0) {
    if (N > 0) SAO_CUDA_TRY(cudaMemsetAsync(adv, 0, sizeof(float) * size_t(N), s));
    return SAO_OK;
  }
  // chunk_first (written by the group pass for the broadcast) and the flag
  // start at zero, then the flag is set to 1 (sorted until shown otherwise)
  SAO_CUDA_TRY(cudaMemsetAsync(chunk_first, 0, size_t(reinterpret_cast<char *>(sorted + 1) -
                                                       reinterpret_cast<char *>(chunk_first)), s));
  SAO_CUDA_TRY(cudaMemsetAsync(sorted, 1, 1, s));  // the int 1
  const int nchunks = int((N + kSegChunk - 1) / kSegChunk);
  int slot = launch_begin("group_advantages", s);
  group_sorted_kernel<<<unsigned((B + 255) / 256), 256, 0, s>>>(gid, B, sorted);
  group_norm_kernel<<<unsigned((B + 7) / 8), 256, 0, s>>>(rewards, gid, B, eps, sorted, a_traj, cu, N, nchunks,
                                                          chunk_first);
  SAO_TRY(launch_end(slot, s));
  return broadcast_launch(a_traj, m, cu, B, N, chunk_first, adv, s);
}

sao_status running_mean_launch(const float *rewards, const int32_t *pid, int32_t B, int32_t P, float *history,
                               int64_t *seen, int32_t window, const uint8_t *m, const int32_t *cu, int64_t N,
                               float *adv, void *ws_body, size_t body_bytes, cudaStream_t s) {
  Carver c(ws_body, body_bytes);
  float *a_traj = c.take<float>(size_t(B) + 1);
  long long *rec = c.take<long long>(size_t(B) + 1);
  int *chunk_first = c.take<int>(size_t((N + kSegChunk - 1) / kSegChunk) + 1);
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the running-mean baseline");
  if (B == 0) {
    if (N > 0) SAO_CUDA_TRY(cudaMemsetAsync(adv, 0, sizeof(float) * size_t(N), s));
    return SAO_OK;
  }
  // the rank table, when the prompt ids are few enough and it fits in the rest of the workspace
  const int nblk = (B + kRankBlock - 1) / kRankBlock;
  int *table = nullptr, *rank = nullptr;
  if (P <= kRankMaxPrompts) {
    Carver t = c;
    int *tab = t.take<int>(size_t(nblk + 1) * size_t(P));
    int *rk = t.take<int>(size_t(B));
    if (t.ok()) {
      table = tab;
      rank = rk;
    }
  }
  const int nchunks = int((N + kSegChunk - 1) / kSegChunk);
  // chunk_first (written by the per-trajectory pass for the broadcast) starts at zero
  SAO_CUDA_TRY(cudaMemsetAsync(chunk_first, 0, sizeof(int) * (size_t(nchunks) + 1), s));
  int slot = launch_begin("running_mean_advantages", s);
  if (table) {
    rank_count_kernel<<<unsigned(nblk), 256, 0, s>>>(pid, B, P, table);
    rank_scan_kernel<<<unsigned((P + 7) / 8), 256, 0, s>>>(table, nblk, P);
  }
  const unsigned g = unsigned((B + 7) / 8);  // a warp per trajectory
  running_mean_kernel<<<g, 256, 0, s>>>(rewards, pid, B, P, table, history,
                                        reinterpret_cast<const long long *>(seen), window, a_traj, rec, rank, cu,
                                        N, nchunks, chunk_first);
  running_mean_record_kernel<<<g, 256, 0, s>>>(rewards, pid, B, P, table ? table + int64_t(nblk) * P : nullptr,
                                               rank, rec, history, reinterpret_cast<long long *>(seen), window);
  SAO_TRY(launch_end(slot, s));
  return broadcast_launch(a_traj, m, cu, B, N, chunk_first, adv, s);
}

}  // namespace sao
