// Step-level GAE (App. A.1): the advantage is computed per step (one
// conversation turn = a maximal run of action tokens inside a trajectory) and
// broadcast to the step's tokens.
//
//   1. flag trajectory starts (a bit mask), then step starts (an action token
//      that opens a trajectory or follows a non-action token); a count pass,
//      a scan and a scatter pass give the ordered step list with each step's
//      token range (count on the device) and per-block step offsets;
//   2. a warp takes 32 consecutive steps, one per lane: a lane sums its own
//      step when it is short (most turns), the warp sums the long ones
//      together (below 2^25 tokens, one warp per step); sums are compensated
//      fp32 pairs (~48 bits), so GB300's slow fp64 pipe is not on this path;
//   3. one warp per trajectory runs the backward GAE over its steps: each
//      lane folds a contiguous block of steps into an affine map, a shuffle
//      scan combines the maps, each lane replays its block (double-float; the
//      length-adaptive lambda is counted in steps);
//   4. step by step, every token gets its step's advantage, value target and
//      value-loss flag (non-action tokens get zeros): a warp writes the token
//      spans of 32 consecutive steps, so no per-token index is stored and the
//      mask is not read again.
#include <stdint.h>

#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {
namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerBlock = 4096;       // tokens per block: the unit of the step offsets and of the broadcast
constexpr int kCountRows = 16384;         // tokens per CTA of the count and scatter passes (4 blocks)
constexpr int kTokensPerThread = kCountRows / kThreads;  // 64: four 16-byte loads in flight
constexpr int kSubBlocks = kCountRows / kRowsPerBlock;
constexpr int kWarpsPerBlock = kRowsPerBlock / kTokensPerThread / 32;  // 2
constexpr int kShortStep = 32;  // a step this long or shorter is summed by one lane
constexpr int64_t kWarpPerStepBelow = int64_t(1) << 25;  // fewer tokens than this: one warp per step

// Trajectory starts as a bit mask over the tokens (bit t & 31 of word t >> 5).
__global__ void mark_traj_starts(const int32_t *cu, int B, int64_t N, uint32_t *tsb) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int64_t t = cu[b];
  if (t >= 0 && t < N && cu[b + 1] > t) atomicOr(tsb + (t >> 5), 1u << (t & 31));
}
// Trajectory-start bits of the n (32, 4 or 1) tokens from t0, a multiple of
// n (zero past N).
__device__ __forceinline__ uint32_t ts_bits(const uint32_t *tsb, int64_t N, int64_t t0, int n) {
  const uint32_t mask = n >= 32 ? 0xFFFFFFFFu : (1u << n) - 1u;
  return t0 < N ? (__ldg(tsb + (t0 >> 5)) >> (t0 & 31)) & mask : 0u;
}

// Bit i set when byte i of x is non-zero (i = 0..3).
__device__ __forceinline__ uint32_t nz4(uint32_t x) {
  const uint32_t h = (((x & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | x) & 0x80808080u;
  return (h * 0x00204081u) >> 28;
}

// Step starts among the 64 tokens t0 .. t0+63, t0 a multiple of 64 (bit i:
// token t0+i opens a step: an action token that opens a trajectory or
// follows a non-action token), their action flags and trajectory starts.
// Four 16-byte loads in flight when the run is in range and aligned, byte
// loads otherwise.
__device__ __forceinline__ uint64_t step_starts64(const uint8_t *m, const uint32_t *tsb, int64_t N, int64_t t0,
                                                  uint64_t &act, uint64_t &tstart) {
  uint64_t M = 0;
  const uint64_t T = uint64_t(ts_bits(tsb, N, t0, 32)) | uint64_t(ts_bits(tsb, N, t0 + 32, 32)) << 32;
  if (t0 + 64 <= N && (reinterpret_cast<uintptr_t>(m) & 15u) == 0) {
    uint4 mv[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) mv[k] = __ldg(reinterpret_cast<const uint4 *>(m + t0) + k);
#pragma unroll
    for (int k = 0; k < 4; ++k)
      M |= uint64_t(nz4(mv[k].x) | nz4(mv[k].y) << 4 | nz4(mv[k].z) << 8 | nz4(mv[k].w) << 12) << (16 * k);
  } else {
    for (int i = 0; i < 64; ++i)
      if (t0 + i < N) M |= uint64_t(m[t0 + i] != 0) << i;
  }
  const uint64_t prev = (M << 1) | uint64_t(t0 > 0 && t0 - 1 < N && m[t0 - 1] != 0);  // bit i: token t0+i-1 acts
  act = M;
  tstart = T;
  return M & (T | ~prev);
}

// Step starts per CTA of kCountRows tokens, each thread 64 consecutive tokens.
__global__ void __launch_bounds__(kThreads) step_count_kernel(const uint8_t *m, const uint32_t *ts, int64_t N,
                                                              int *cta_count) {
  const int64_t t0 = int64_t(blockIdx.x) * kCountRows + int64_t(threadIdx.x) * kTokensPerThread;
  uint64_t act, tst;
  int c = t0 < N ? __popcll(step_starts64(m, ts, N, t0, act, tst)) : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __shared__ int sh[kThreads / 32];
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < kThreads / 32; ++w) s += sh[w];
    cta_count[blockIdx.x] = s;
  }
}
static_assert(kTokensPerThread == 64 && kWarpsPerBlock * 32 * kTokensPerThread == kRowsPerBlock,
              "64 tokens per thread, whole warps per block");

// Exclusive scan of the per-block step counts in place (one CTA of 1024
// threads). Thread i owns a run of `per` consecutive counts, `per` a multiple
// of 8, so each 8-count piece is two aligned 16-byte loads and a thread's
// pieces are all in flight at once; warp shuffles and one shared-memory row
// of warp totals scan the thread sums.
constexpr int kScanPiece = 8;

__device__ __forceinline__ void load_piece(const int *p, int b, int nblocks, int (&v)[kScanPiece]) {
  if (b + kScanPiece <= nblocks && (reinterpret_cast<uintptr_t>(p) & 15u) == 0) {
    const int4 x = *reinterpret_cast<const int4 *>(p + b);
    const int4 y = *reinterpret_cast<const int4 *>(p + b + 4);
    v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w;
    v[4] = y.x; v[5] = y.y; v[6] = y.z; v[7] = y.w;
  } else {
#pragma unroll
    for (int k = 0; k < kScanPiece; ++k) v[k] = b + k < nblocks ? p[b + k] : 0;
  }
}

__global__ void __launch_bounds__(1024) step_scan_kernel(int *block_count, int nblocks, int *total) {
  __shared__ int sh[32];
  const int per = ((nblocks + 1023) / 1024 + kScanPiece - 1) / kScanPiece * kScanPiece;
  const int b0 = threadIdx.x * per;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int s = 0;
#pragma unroll 4
  for (int i = 0; i < per; i += kScanPiece) {
    int v[kScanPiece];
    load_piece(block_count, b0 + i, nblocks, v);
#pragma unroll
    for (int k = 0; k < kScanPiece; ++k) s += v[k];
  }
  int x = s;  // inclusive scan of the thread sums within the warp
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = sh[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;  // inclusive over warps
  }
  __syncthreads();
  int run = (warp ? sh[warp - 1] : 0) + x - s;
#pragma unroll 4
  for (int i = 0; i < per; i += kScanPiece) {
    int v[kScanPiece];
    load_piece(block_count, b0 + i, nblocks, v);
#pragma unroll
    for (int k = 0; k < kScanPiece; ++k) {
      const int b = b0 + i + k;
      if (b < nblocks) block_count[b] = run;
      run += v[k];
    }
  }
  if (threadIdx.x == 1023) *total = sh[31];
}

// Ordered step list with each step's first and one-past-last token.
// Also writes, per block of kRowsPerBlock tokens, the steps opened before it
// (the offsets the step search and the broadcast use).
__global__ void __launch_bounds__(kThreads) step_scatter_kernel(const uint8_t *m, const uint32_t *ts, int64_t N,
                                                                const int *cta_offset, int nblocks,
                                                                int *block_offset, int *step_first,
                                                                int *step_end) {
  const int64_t t0 = int64_t(blockIdx.x) * kCountRows + int64_t(threadIdx.x) * kTokensPerThread;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint64_t act = 0, st = 0, tst = 0;
  if (t0 < N) st = step_starts64(m, ts, N, t0, act, tst);
  // does token t0+64 continue a step? (an action token that opens no trajectory)
  const uint32_t lo_act = uint32_t(act), lo_tst = uint32_t(tst);
  uint32_t nact = __shfl_down_sync(0xffffffffu, lo_act, 1), ntst = __shfl_down_sync(0xffffffffu, lo_tst, 1);
  if (lane == 31) {
    const int64_t u = t0 + kTokensPerThread;
    nact = (u < N && m[u] != 0) ? 1u : 0u;
    ntst = ts_bits(ts, N, u, 1);
  }
  const uint64_t cont_next = (nact & ~ntst) & 1u;
  // bit i: token t0+i+1 continues the step; last: token t0+i is a step's last token
  const uint64_t cont = ((act & ~tst) >> 1) | (cont_next << 63);
  const uint64_t last = act & ~cont;
  const int c = __popcll(st);
  // exclusive prefix of the counts over the block
  int x = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __shared__ int sh[kThreads / 32];
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  const int cta0 = cta_offset[blockIdx.x];
  if (threadIdx.x < kSubBlocks) {
    const int blk = blockIdx.x * kSubBlocks + threadIdx.x;
    int o = cta0;
    for (int w = 0; w < threadIdx.x * kWarpsPerBlock; ++w) o += sh[w];
    if (blk < nblocks) block_offset[blk] = o;
  }
  if (t0 >= N) return;
  int before = 0;
  for (int w = 0; w < warp; ++w) before += sh[w];
  const int base = cta0 + before + x - c;  // steps opened before token t0
  int k = base;
  uint64_t bits = st | last;
  while (bits) {
    const int i = __ffsll(static_cast<long long>(bits)) - 1;
    bits &= bits - 1;
    if ((st >> i) & 1u) step_first[k++] = int(t0 + i);
    if ((last >> i) & 1u) step_end[k - 1] = int(t0 + i + 1);
  }
}

// Compensated fp32 accumulator (Knuth two-sum).
struct Acc2 {
  float hi = 0.f, lo = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float s = __fadd_rn(hi, x);
    const float bb = __fsub_rn(s, hi);
    lo = __fadd_rn(lo, __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(x, bb)));
    hi = s;
  }
  __device__ __forceinline__ void add(const Acc2 &o) {
    add(o.hi);
    lo = __fadd_rn(lo, o.lo);
  }
};

// ---------------------------------------------------------------------------
// double-float arithmetic (fp32 pairs, ~48 bits): GB300's fp64 pipe is far
// slower than its fp32 one, and these recurrences run over millions of steps
// ---------------------------------------------------------------------------
struct dd {
  float hi, lo;
};
__device__ __forceinline__ dd dd_quick(float a, float b) {  // |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ dd dd_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
__device__ __forceinline__ dd dd_add(dd x, dd y) {
  const dd s = dd_two_sum(x.hi, y.hi);
  return dd_quick(s.hi, __fadd_rn(s.lo, __fadd_rn(x.lo, y.lo)));
}
__device__ __forceinline__ dd dd_mul(dd x, dd y) {
  const float p = __fmul_rn(x.hi, y.hi);
  float e = __fmaf_rn(x.hi, y.hi, -p);
  e = __fmaf_rn(x.hi, y.lo, e);
  e = __fmaf_rn(x.lo, y.hi, e);
  return dd_quick(p, e);
}
__device__ __forceinline__ dd dd_neg(dd x) { return {-x.hi, -x.lo}; }
__device__ __forceinline__ dd dd_from_double(double x) {
  const float hi = float(x);
  return {hi, float(x - double(hi))};
}
__device__ __forceinline__ float dd_round(dd x) { return __fadd_rn(x.hi, x.lo); }

// Step value V(S) as a double-float: the mean of a compensated sum over n tokens.
__device__ __forceinline__ float2 acc_mean(const Acc2 &a, int n) {
  const float fn = float(n);
  const float q = __fdiv_rn(a.hi, fn);
  const float r = __fadd_rn(__fmaf_rn(-q, fn, a.hi), a.lo);
  const dd m = dd_quick(q, __fdiv_rn(r, fn));
  return make_float2(m.hi, m.lo);
}

// A warp takes 32 consecutive steps, one per lane: a lane sums its own step
// when it is short (8 independent loads at a time), the warp sums the long
// ones together; below kWarpPerStepBelow tokens, a warp takes one step. Step
// ranges come from the scatter pass, so no load waits on another. (Copying
// the warp's span of values into shared memory first, for contiguous loads,
// measured 3x slower: the copy exposes a load latency per 32 values, while
// the steps' own loads already fall in a few nearby lines.)
template <bool kWarpPerStep>
__global__ void __launch_bounds__(kThreads) step_reduce_kernel(const float *values, const int *step_first,
                                                               const int *step_end, const int *nsteps, int mode,
                                                               float2 *sv) {
  const int lane = threadIdx.x & 31;
  const int S = *nsteps;
  const int nwarps = (gridDim.x * kThreads) >> 5;
  if (kWarpPerStep && mode != SAO_STEP_LAST) {
    // few steps: one warp per step, so every SM has work (the mode depends
    // on N alone, so every device gives the same bits)
    for (int s = (blockIdx.x * kThreads + threadIdx.x) >> 5; s < S; s += nwarps) {
      const int f = step_first[s], e = step_end[s];
      Acc2 part;
      for (int t = f + lane; t < e; t += 256) {
        float x[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) x[k] = t + 32 * k < e ? values[t + 32 * k] : 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (t + 32 * k < e) part.add(x[k]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        Acc2 other;
        other.hi = __shfl_xor_sync(0xffffffffu, part.hi, o);
        other.lo = __shfl_xor_sync(0xffffffffu, part.lo, o);
        part.add(other);
      }
      if (lane == 0) sv[s] = acc_mean(part, e - f);
    }
    return;
  }
  // the next group's step ranges are loaded while this group is summed
  int g = (blockIdx.x * kThreads + threadIdx.x) >> 5;
  int nfirst = g * 32 + lane < S ? step_first[g * 32 + lane] : 0;
  int nend = g * 32 + lane < S ? step_end[g * 32 + lane] : 0;
  for (; g * 32 < S; g += nwarps) {
    const int s = g * 32 + lane;
    const bool own = s < S;
    const int first = nfirst, end = nend;
    const int sn = (g + nwarps) * 32 + lane;
    if (sn < S) {
      nfirst = step_first[sn];
      nend = step_end[sn];
    }
    if (mode == SAO_STEP_LAST) {  // the value of the step's last token
      if (own) sv[s] = make_float2(values[end - 1], 0.f);
      continue;
    }
    const bool shortstep = own && end - first <= kShortStep;
    Acc2 acc;
    if (shortstep) {
      // 8 tokens at a time, the loads of a group (the ragged last one too)
      // issued before its adds, which keep the token order
      for (int t = first; t < end; t += 8) {
        float x[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) x[k] = t + k < end ? values[t + k] : 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (t + k < end) acc.add(x[k]);
      }
    }
    unsigned longs = __ballot_sync(0xffffffffu, own && !shortstep);
    while (longs) {
      const int src = __ffs(longs) - 1;
      longs &= longs - 1;
      const int f = __shfl_sync(0xffffffffu, first, src), e = __shfl_sync(0xffffffffu, end, src);
      Acc2 part;
      // a lane's tokens f + lane, f + lane + 32, ... in order, eight loads at a time
      for (int t = f + lane; t < e; t += 256) {
        float x[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) x[k] = t + 32 * k < e ? values[t + 32 * k] : 0.f;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (t + 32 * k < e) part.add(x[k]);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        Acc2 other;
        other.hi = __shfl_xor_sync(0xffffffffu, part.hi, o);
        other.lo = __shfl_xor_sync(0xffffffffu, part.lo, o);
        part.add(other);
      }
      if (lane == src) acc = part;
    }
    if (own) sv[s] = acc_mean(acc, end - first);
  }
}

// Affine map of a block of steps: A_left = p * A_right + c.
struct StepMap {
  dd p, c;
};
__device__ __forceinline__ StepMap compose_steps(const StepMap &x, const StepMap &y) {  // x left of y
  return {dd_mul(x.p, y.p), dd_add(dd_mul(x.p, y.c), x.c)};
}
__device__ __forceinline__ dd dd_shfl_down(dd x, int d) {
  return {__shfl_down_sync(0xffffffffu, x.hi, d), __shfl_down_sync(0xffffffffu, x.lo, d)};
}

constexpr int kGaeWarps = 4;  // warps (trajectories) per CTA of step_gae_kernel
constexpr int kStepGroup = 8; // step values a lane loads ahead of its recursion

// One warp per trajectory: lane l folds steps [s0 + l*c, s0 + (l+1)*c) into
// maps for the policy (a = gamma*lambda_b) and the critic (a = gamma*lambda_c),
// a shuffle scan gives each lane the advantages to the right of its block, and
// the lane replays its block. Both passes walk the block backwards in groups
// of kStepGroup steps whose values are loaded before the group's recursion, so
// a long trajectory (thousands of steps per lane) waits for one load latency
// per group, not per step.
// kCrit false: gamma = lambda_critic = 1, where the critic's return telescopes
// to the trajectory's reward R on every step, so only the policy recursion runs.
template <bool kCrit>
__global__ void __launch_bounds__(32 * kGaeWarps) step_gae_kernel(const float *rewards, const int32_t *cu, int B,
                                                                  int64_t N, const int *step_first,
                                                                  const int *block_offset, int nblocks,
                                                                  const int *nsteps, const float2 *sv, float gamma,
                                                                  float lam, float lam_c, float alpha,
                                                                  float2 *out /*[S] (adv, ret)*/) {
  const int lane = threadIdx.x & 31;
  const int b = (blockIdx.x * (32 * kGaeWarps) + threadIdx.x) >> 5;
  if (b >= B) return;
  const int S = *nsteps;
  // steps of trajectory b: those whose first token lies in [cu[b], cu[b+1]);
  // first step index with step_first >= t by a 33-way warp search, starting
  // from the steps opened before t's 4096-token block and before the next one
  auto lower = [&](int64_t t) {
    if (t >= N) return S;
    const int blk = int(t / kRowsPerBlock);
    int lo = block_offset[blk];
    int hi = blk + 1 < nblocks ? block_offset[blk + 1] : S;  // the answer lies in [lo, hi]
    while (hi - lo > 32) {
      const int p = lo + int(int64_t(hi - lo) * (lane + 1) / 33);  // 32 rising pivots in [lo, hi)
      const unsigned below = __ballot_sync(0xffffffffu, int64_t(step_first[p]) < t);
      const int c = __popc(below);  // pivots below t: lanes 0 .. c-1
      const int nlo = c > 0 ? __shfl_sync(0xffffffffu, p, c - 1) + 1 : lo;
      const int nhi = c < 32 ? __shfl_sync(0xffffffffu, p, c & 31) : hi;
      lo = nlo;
      hi = nhi;
    }
    const bool below = lo + lane < hi && int64_t(step_first[lo + lane]) < t;
    return lo + __popc(__ballot_sync(0xffffffffu, below));
  };
  const int s0 = lower(cu[b]);
  const int s1 = lower(cu[b + 1]);
  const int n = s1 - s0;
  if (n <= 0) return;
  double lb = lam;
  if (alpha > 0.f) {
    lb = 1.0 - 1.0 / (double(alpha) * double(n));
    lb = lb < 0.0 ? 0.0 : (lb > 1.0 ? 1.0 : lb);
  }
  const dd ap = dd_from_double(double(gamma) * lb), ac = dd_from_double(double(gamma) * double(lam_c));
  const dd g = {gamma, 0.f};
  const float R = rewards[b];
  const int c = (n + 31) / 32;
  const int a0 = s0 + lane * c, a1 = min(a0 + c, s1);  // this lane's steps [a0, a1)
  auto value = [&](int i) {
    const float2 v = sv[i];
    return dd{v.x, v.y};
  };
  // delta_i = r_i + gamma v_{i+1} - v_i (the reward only on the trajectory's last step)
  auto delta = [&](int i, dd v, dd v_next) {
    dd d = dd_add(dd_mul(g, v_next), dd_neg(v));
    if (i == s1 - 1) d = dd_add(d, dd{R, 0.f});
    return d;
  };
  const dd zero = {0.f, 0.f}, one = {1.f, 0.f};
  const dd v_after = a1 < s1 ? value(a1) : zero;  // value of the step right after the block
  StepMap mp{one, zero}, mc{one, zero};
  {
    dd v_next = v_after;
    auto fold = [&](int i, float2 vi) {
      const dd v{vi.x, vi.y};
      const dd d = delta(i, v, v_next);
      mp = {dd_mul(ap, mp.p), dd_add(dd_mul(ap, mp.c), d)};
      if constexpr (kCrit) mc = {dd_mul(ac, mc.p), dd_add(dd_mul(ac, mc.c), d)};
      v_next = v;
    };
    int i = a1 - 1;
    for (; i - (kStepGroup - 1) >= a0; i -= kStepGroup) {
      float2 vg[kStepGroup];
#pragma unroll
      for (int k = 0; k < kStepGroup; ++k) vg[k] = sv[i - k];
#pragma unroll
      for (int k = 0; k < kStepGroup; ++k) fold(i - k, vg[k]);
    }
    for (; i >= a0; --i) fold(i, sv[i]);
  }
  // suffix scan over lanes: the maps of lanes l+1 .. 31 applied to A = 0
  StepMap sp = mp, sc = mc;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const StepMap op{dd_shfl_down(sp.p, d), dd_shfl_down(sp.c, d)};
    if (lane + d < 32) sp = compose_steps(sp, op);
    if constexpr (kCrit) {
      const StepMap oc{dd_shfl_down(sc.p, d), dd_shfl_down(sc.c, d)};
      if (lane + d < 32) sc = compose_steps(sc, oc);
    }
  }
  dd Ap = dd_shfl_down(sp.c, 1), Ac = zero;  // advantages of the step right of the block
  if constexpr (kCrit) Ac = dd_shfl_down(sc.c, 1);
  if (lane == 31) Ap = Ac = zero;
  dd v_next = v_after;
  auto replay = [&](int i, float2 vi) {
    const dd v{vi.x, vi.y};
    const dd d = delta(i, v, v_next);
    Ap = dd_add(dd_mul(ap, Ap), d);
    float r = R;
    if constexpr (kCrit) {
      Ac = dd_add(dd_mul(ac, Ac), d);
      r = dd_round(dd_add(Ac, v));
    }
    out[i] = make_float2(dd_round(Ap), r);
    v_next = v;
  };
  int i = a1 - 1;
  for (; i - (kStepGroup - 1) >= a0; i -= kStepGroup) {
    float2 vg[kStepGroup];
#pragma unroll
    for (int k = 0; k < kStepGroup; ++k) vg[k] = sv[i - k];
#pragma unroll
    for (int k = 0; k < kStepGroup; ++k) replay(i - k, vg[k]);
  }
  for (; i >= a0; --i) replay(i, sv[i]);
}

// Every token gets its step's results (non-action tokens get zeros), step by
// step: a warp takes 32 consecutive steps (one per lane: first token, end,
// results) and writes the tokens from its first step's first token to the
// next group's (the steps and the observation tokens after each), or a share
// of those windows when there are fewer groups than warps, in 128-token
// windows with 4 tokens per lane, so every store of the warp is contiguous. A lane finds the step of its tokens by a binary search over the
// 32 first tokens held in the warp's lanes; the first group also writes the
// tokens before the first step. Neither the mask nor the flags are read again.
__device__ __forceinline__ int steps_at_or_before(int F, int t) {  // #{j : F_j <= t}, F_j rising over the lanes
  int pos = 0;
#pragma unroll
  for (int b = 16; b >= 1; b >>= 1) {
    const int f = __shfl_sync(0xffffffffu, F, pos + b - 1);
    if (f <= t) pos += b;
  }
  const int f31 = __shfl_sync(0xffffffffu, F, 31);
  return (pos == 31 && f31 <= t) ? 32 : pos;
}

__global__ void __launch_bounds__(kThreads) step_broadcast_kernel(const int *nsteps, const int *step_first,
                                                                  const int *step_end, const float2 *out, int mode,
                                                                  int64_t N, float *adv, float *ret, uint8_t *vmask) {
  const int lane = threadIdx.x & 31;
  const int S = *nsteps;
  const int ngroups = S > 0 ? (S + 31) / 32 : 1;
  const int nwarps = (gridDim.x * kThreads) >> 5;
  // with fewer groups than warps, each group's windows are shared out over
  // up to 64 warps
  const int parts = max(1, min(64, nwarps / ngroups));
  const bool vout = ((reinterpret_cast<uintptr_t>(adv) | reinterpret_cast<uintptr_t>(ret)) & 15u) == 0 &&
                    (reinterpret_cast<uintptr_t>(vmask) & 3u) == 0;
  const bool last_mode = mode != SAO_STEP_AVERAGE;
  for (int u = (blockIdx.x * kThreads + threadIdx.x) >> 5; u < ngroups * parts; u += nwarps) {
    const int g = u / parts, part = u % parts;
    const int s = g * 32 + lane;
    const bool has = s < S;
    const int F = has ? step_first[s] : INT_MAX;
    const int E = has ? step_end[s] : 0;
    const float2 o = has ? out[s] : make_float2(0.f, 0.f);
    const int lo = g == 0 ? 0 : __shfl_sync(0xffffffffu, F, 0);
    const int hi = (g + 1) * 32 < S ? step_first[(g + 1) * 32] : int(N);  // the group writes [lo, hi)
    const int c0 = lo & ~3;
    const int nwin = (hi - c0 + 127) / 128, per = (nwin + parts - 1) / parts;
    const int w1 = min(nwin, (part + 1) * per);
    for (int win = part * per; win < w1; ++win) {
      const int t4 = c0 + 128 * win + 4 * lane;
      float a[4], r[4];
      uint8_t k[4];
      const int j0 = steps_at_or_before(F, t4) - 1;  // step of token t4 in the group (-1: before it)
      const int fn = __shfl_sync(0xffffffffu, F, j0 + 1 < 32 ? j0 + 1 : 31);
      const int next = j0 + 1 < 32 ? fn : INT_MAX;  // first token of the step after j0 in the group
      if (__all_sync(0xffffffffu, next > t4 + 3)) {
        // the lane's 4 tokens lie in one step's tokens and the gap after them
        const int src = j0 < 0 ? 0 : j0;
        const float sa = __shfl_sync(0xffffffffu, o.x, src), sr = __shfl_sync(0xffffffffu, o.y, src);
        const int se = __shfl_sync(0xffffffffu, E, src);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const bool in = j0 >= 0 && t4 + i < se;
          a[i] = in ? sa : 0.f;
          r[i] = in ? sr : 0.f;
          k[i] = (in && (!last_mode || t4 + i == se - 1)) ? 1 : 0;
        }
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int j = steps_at_or_before(F, t4 + i) - 1;
          const int src = j < 0 ? 0 : j;
          const float sa = __shfl_sync(0xffffffffu, o.x, src), sr = __shfl_sync(0xffffffffu, o.y, src);
          const int se = __shfl_sync(0xffffffffu, E, src);
          const bool in = j >= 0 && t4 + i < se;
          a[i] = in ? sa : 0.f;
          r[i] = in ? sr : 0.f;
          k[i] = (in && (!last_mode || t4 + i == se - 1)) ? 1 : 0;
        }
      }
      if (vout && t4 >= lo && t4 + 3 < hi) {
        __stcs(reinterpret_cast<float4 *>(adv + t4), make_float4(a[0], a[1], a[2], a[3]));
        __stcs(reinterpret_cast<float4 *>(ret + t4), make_float4(r[0], r[1], r[2], r[3]));
        if (vmask) *reinterpret_cast<uchar4 *>(vmask + t4) = make_uchar4(k[0], k[1], k[2], k[3]);
      } else {
        for (int i = 0; i < 4; ++i) {
          const int t = t4 + i;
          if (t < lo || t >= hi) continue;
          adv[t] = a[i];
          ret[t] = r[i];
          if (vmask) vmask[t] = k[i];
        }
      }
    }
  }
}

}  // namespace

size_t step_gae_ws_bytes(int64_t N, int64_t B) {
  (void)B;
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t nctas = (N + kCountRows - 1) / kCountRows;
  return round256(sizeof(uint32_t) * size_t((N + 31) / 32)) + round256(sizeof(int) * (nctas + 1)) +
         round256(sizeof(int) * (nblocks + 1)) + round256(sizeof(int) * 4) +
         round256(sizeof(int) * N) + round256(sizeof(int) * N) + round256(sizeof(float2) * N) +
         round256(sizeof(float2) * N);
}

sao_status step_gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu, int32_t B,
                           int64_t N, float gamma, float lam, float lam_c, float alpha, int mode, float *adv,
                           float *ret, uint8_t *vmask, void *ws_body, size_t body_bytes, cudaStream_t s) {
  if (N == 0) return SAO_OK;
  // token indices are int32 here, with room for a 128-token window past N
  if (N > int64_t(INT_MAX) - 256) return fail(SAO_ERR_SHAPE, "too many tokens for the step-level advantages");
  const int64_t nblocks = (N + kRowsPerBlock - 1) / kRowsPerBlock;
  Carver c(ws_body, body_bytes);
  const size_t ts_words = size_t((N + 31) / 32);
  uint32_t *ts = c.take<uint32_t>(ts_words);
  const int64_t nctas = (N + kCountRows - 1) / kCountRows;
  int *cta = c.take<int>(size_t(nctas) + 1);
  int *block = c.take<int>(size_t(nblocks) + 1);
  int *nsteps = c.take<int>(4);
  int *step_first = c.take<int>(size_t(N));
  int *step_end = c.take<int>(size_t(N));
  float2 *sv = c.take<float2>(size_t(N));
  float2 *out = c.take<float2>(size_t(N));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the step-level advantages");
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  SAO_CUDA_TRY(cudaMemsetAsync(ts, 0, sizeof(uint32_t) * ts_words, s));
  int slot = launch_begin("step_gae_segments", s);
  mark_traj_starts<<<unsigned((B + 255) / 256), 256, 0, s>>>(cu, B, N, ts);
  const unsigned count_grid = unsigned((N + kCountRows - 1) / kCountRows);
  step_count_kernel<<<count_grid, kThreads, 0, s>>>(m, ts, N, cta);
  step_scan_kernel<<<1, 1024, 0, s>>>(cta, int(nctas), nsteps);
  step_scatter_kernel<<<count_grid, kThreads, 0, s>>>(m, ts, N, cta, int(nblocks), block, step_first, step_end);
  SAO_TRY(launch_end(slot, s));
  const unsigned warps_grid = unsigned(di.sm_count * 8);
  slot = launch_begin("step_gae_reduce", s);
  auto reduce = N < kWarpPerStepBelow ? step_reduce_kernel<true> : step_reduce_kernel<false>;
  reduce<<<warps_grid, kThreads, 0, s>>>(values, step_first, step_end, nsteps, mode, sv);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("step_gae_scan", s);
  auto scan = (gamma == 1.f && lam_c == 1.f) ? step_gae_kernel<false> : step_gae_kernel<true>;
  scan<<<unsigned((int64_t(B) + kGaeWarps - 1) / kGaeWarps), 32 * kGaeWarps, 0, s>>>(
      rewards, cu, B, N, step_first, block, int(nblocks), nsteps, sv, gamma, lam, lam_c, alpha, out);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("step_gae_broadcast", s);
  step_broadcast_kernel<<<warps_grid, kThreads, 0, s>>>(nsteps, step_first, step_end, out, mode, N, adv, ret, vmask);
  return launch_end(slot, s);
}

}  // namespace sao
