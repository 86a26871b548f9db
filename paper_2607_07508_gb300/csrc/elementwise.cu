// Policy loss (Eq. 1-3, §3.1), the decoupled three-policy objective that DIS
// simplifies (§3.1) and value loss (Preliminaries, §4.4) kernels.
//
// Both are HBM-bound streams over the packed tokens: 16-byte vector loads of
// four tokens at a time, a grid of a few CTAs per SM striding over the input,
// per-CTA partial sums written to the workspace and a one-CTA finaliser that
// adds the partials in a fixed order, so every result is deterministic.
// When the caller does not pass its own normaliser, a first pass counts the
// action tokens (1 byte per token) so the per-token outputs can be scaled in
// the same pass that computes them.
#include <stdint.h>

#include "sao_common.cuh"
#include "sao_internal.h"

namespace sao {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ long long warp_sum(long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the CTA in a fixed tree order; result valid in thread 0.
template <class T>
__device__ T block_sum(T v) {
  __shared__ T sh[kThreads / 32];
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) sh[w] = v;
  __syncthreads();
  T r = 0;
  if (w == 0) {
    r = (l < kThreads / 32) ? sh[l] : T(0);
    r = warp_sum(r);
  }
  __syncthreads();
  return r;
}

// ---------------------------------------------------------------------------
// action-token count (n_valid)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) count_mask_kernel(const uint8_t *__restrict__ m,
                                                             int64_t N, long long *partial) {
  long long c = 0;
  const int64_t tid = int64_t(blockIdx.x) * kThreads + threadIdx.x;
  const int64_t stride = int64_t(gridDim.x) * kThreads;
  const bool vec = (reinterpret_cast<uintptr_t>(m) & 15u) == 0;
  int64_t done = 0;
  if (vec) {
    const int64_t n16 = N / 16;
    const uint4 *m16 = reinterpret_cast<const uint4 *>(m);
    // a mask byte is 0 or non-zero; count non-zero bytes
    auto count16 = [](const uint4 q) {
      const uint32_t w[4] = {q.x, q.y, q.z, q.w};
      int n = 0;
#pragma unroll
      for (int k = 0; k < 4; ++k) n += __popc(((w[k] & 0x7f7f7f7fu) + 0x7f7f7f7fu | w[k]) & 0x80808080u);
      return n;
    };
    int64_t i = tid;
    // four independent 16-byte loads in flight per thread
    for (; i + 3 * stride < n16; i += 4 * stride) {
      uint4 q[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) q[u] = __ldg(m16 + i + u * stride);
#pragma unroll
      for (int u = 0; u < 4; ++u) c += count16(q[u]);
    }
    for (; i < n16; i += stride) c += count16(__ldg(m16 + i));
    done = n16 * 16;
  }
  for (int64_t i = done + tid; i < N; i += stride) c += (m[i] != 0);
  c = block_sum(c);
  if (threadIdx.x == 0) partial[blockIdx.x] = c;
}

// Every CTA of the consumer kernel sums the same partials in the same order.
__device__ __forceinline__ long long total_of(const long long *partial, int n) {
  __shared__ long long sh_total;
  long long c = 0;
  for (int i = threadIdx.x; i < n; i += kThreads) c += partial[i];
  c = block_sum(c);
  if (threadIdx.x == 0) sh_total = c;
  __syncthreads();
  return sh_total;
}

// ---------------------------------------------------------------------------
// policy loss, Eq. 1-3
// ---------------------------------------------------------------------------
struct PLToken {
  float coef;
  uint8_t flag;
};

// One token: ratio (Eq. 2), strict mask (Eq. 3), contribution to the
// surrogate -f(r) A and its derivative with f detached.
__device__ __forceinline__ PLToken pl_token(float lp, float old, float a, uint8_t m, float lo,
                                            float hi, float inv_n, float &contrib, int &n_low,
                                            int &n_high, int &n_nonfin) {
  PLToken t{0.f, SAO_FLAG_NOT_ACTION};
  if (!m) return t;
  const float d = lp - old;
  if (!isfinite(d) || !isfinite(a)) {
    t.flag = SAO_FLAG_NONFINITE;
    n_nonfin++;
    return t;
  }
  const float r = expf(d);
  if (r <= lo) {
    t.flag = SAO_FLAG_LOW;
    n_low++;
  } else if (r >= hi) {
    t.flag = SAO_FLAG_HIGH;
    n_high++;
  } else {
    const float c = r * a;
    contrib += c;
    t.flag = SAO_FLAG_IN;
    t.coef = -c * inv_n;
  }
  return t;
}

struct PLArgs {
  const float *logp, *old, *adv;
  const uint8_t *m;
  int64_t N;
  float lo, hi;
  int64_t n_norm;
  const long long *cnt_partial;
  int n_cnt;
  long long *act_out;  // fwd with n_norm > 0: per-CTA action-token counts (no count pass ran)
  float *coef;       // may be null
  uint8_t *flags;    // may be null
  const float *grad_scale;  // bwd: device scalar; fwd: null
  double *loss_partial;
  long long *cnt3_partial;  // [3][grid]
};

__device__ __forceinline__ int nonzero4(uchar4 m) {
  return (m.x != 0) + (m.y != 0) + (m.z != 0) + (m.w != 0);
}

template <bool kBwd>
__global__ void __launch_bounds__(kThreads) policy_loss_kernel(PLArgs a) {
  int64_t n = a.n_norm;
  if (n <= 0) n = total_of(a.cnt_partial, a.n_cnt);
  const float inv_n = n > 0 ? float(1.0 / double(n)) : 0.f;
  const float gscale = kBwd ? __ldg(a.grad_scale) : 1.f;
  double acc = 0.0;
  int n_low = 0, n_high = 0, n_nonfin = 0, n_act = 0;

  const int64_t tid = int64_t(blockIdx.x) * kThreads + threadIdx.x;
  const int64_t stride = int64_t(gridDim.x) * kThreads;
  const bool vec = aligned16_dev(a.logp) && aligned16_dev(a.old) && aligned16_dev(a.adv) &&
                   ((reinterpret_cast<uintptr_t>(a.m) & 3u) == 0) &&
                   (a.coef == nullptr || aligned16_dev(a.coef)) &&
                   (a.flags == nullptr || (reinterpret_cast<uintptr_t>(a.flags) & 3u) == 0);
  int64_t done = 0;
  if (vec) {
    const int64_t n4 = a.N / 4;
    for (int64_t i = tid; i < n4; i += stride) {
      const float4 lp = __ldg(reinterpret_cast<const float4 *>(a.logp) + i);
      const float4 od = __ldg(reinterpret_cast<const float4 *>(a.old) + i);
      const float4 ad = __ldg(reinterpret_cast<const float4 *>(a.adv) + i);
      const uchar4 mk = __ldg(reinterpret_cast<const uchar4 *>(a.m) + i);
      if (!kBwd) n_act += nonzero4(mk);
      float contrib = 0.f;
      PLToken t0 = pl_token(lp.x, od.x, ad.x, mk.x, a.lo, a.hi, inv_n, contrib, n_low, n_high, n_nonfin);
      PLToken t1 = pl_token(lp.y, od.y, ad.y, mk.y, a.lo, a.hi, inv_n, contrib, n_low, n_high, n_nonfin);
      PLToken t2 = pl_token(lp.z, od.z, ad.z, mk.z, a.lo, a.hi, inv_n, contrib, n_low, n_high, n_nonfin);
      PLToken t3 = pl_token(lp.w, od.w, ad.w, mk.w, a.lo, a.hi, inv_n, contrib, n_low, n_high, n_nonfin);
      acc += double(contrib);
      if (a.coef)
        reinterpret_cast<float4 *>(a.coef)[i] =
            make_float4(t0.coef * gscale, t1.coef * gscale, t2.coef * gscale, t3.coef * gscale);
      if (a.flags) reinterpret_cast<uchar4 *>(a.flags)[i] = make_uchar4(t0.flag, t1.flag, t2.flag, t3.flag);
    }
    done = n4 * 4;
  }
  for (int64_t i = done + tid; i < a.N; i += stride) {
    float contrib = 0.f;
    const uint8_t mi = __ldg(a.m + i);
    if (!kBwd) n_act += mi != 0;
    PLToken t = pl_token(__ldg(a.logp + i), __ldg(a.old + i), __ldg(a.adv + i), mi, a.lo,
                         a.hi, inv_n, contrib, n_low, n_high, n_nonfin);
    acc += double(contrib);
    if (a.coef) a.coef[i] = t.coef * gscale;
    if (a.flags) a.flags[i] = t.flag;
  }
  if (kBwd) return;
  acc = block_sum(acc);
  long long l = block_sum((long long)n_low);
  long long h = block_sum((long long)n_high);
  long long f = block_sum((long long)n_nonfin);
  const long long na = a.act_out ? block_sum((long long)n_act) : 0;
  if (threadIdx.x == 0) {
    if (a.act_out) a.act_out[blockIdx.x] = na;
    a.loss_partial[blockIdx.x] = acc;
    a.cnt3_partial[blockIdx.x] = l;
    a.cnt3_partial[gridDim.x + blockIdx.x] = h;
    a.cnt3_partial[2 * gridDim.x + blockIdx.x] = f;
  }
}

__global__ void __launch_bounds__(kThreads) policy_loss_finalize(
    const double *loss_partial, const long long *cnt3_partial, int grid, const long long *cnt_partial,
    int n_cnt, int64_t n_norm, float *loss, int64_t *counts) {
  const long long n_valid = total_of(cnt_partial, n_cnt);
  double s = 0.0;
  long long l = 0, h = 0, f = 0;
  for (int i = threadIdx.x; i < grid; i += kThreads) {
    s += loss_partial[i];
    l += cnt3_partial[i];
    h += cnt3_partial[grid + i];
    f += cnt3_partial[2 * grid + i];
  }
  s = block_sum(s);
  l = block_sum(l);
  h = block_sum(h);
  f = block_sum(f);
  if (threadIdx.x == 0) {
    const long long n = n_norm > 0 ? n_norm : n_valid;
    if (loss) *loss = n > 0 ? float(-s / double(n)) : 0.f;
    if (counts) {
      counts[0] = n_valid;
      counts[1] = l;
      counts[2] = h;
      counts[3] = f;
    }
  }
}

// ---------------------------------------------------------------------------
// decoupled three-policy objective (§3.1)
// ---------------------------------------------------------------------------
struct DLArgs {
  const float *logp, *prox, *roll, *adv;
  const uint8_t *m;
  int64_t N;
  float lo, hi, wlo, whi;
  int64_t n_norm;
  const long long *cnt_partial;
  int n_cnt;
  long long *act_out;  // fwd with n_norm > 0: per-CTA action-token counts (no count pass ran)
  float *coef;              // may be null
  uint8_t *flags;           // may be null
  const float *grad_scale;  // bwd: device scalar; fwd: null
  double *loss_partial;
  long long *cnt5_partial;  // [5][grid]
};

struct DLCounts {
  int low = 0, high = 0, nonfin = 0, wlow = 0, whigh = 0;
};

// One token: the mismatch weight w = pi_old/pi_rollout must lie strictly
// inside (wlo, whi); then the clipped surrogate of r = pi_theta/pi_old, scaled
// by w. Adds the token's -loss contribution to `contrib`.
__device__ __forceinline__ PLToken dl_token(float lp, float px, float ro, float a, uint8_t m, const DLArgs &A,
                                            float inv_n, float &contrib, DLCounts &c) {
  PLToken t{0.f, SAO_FLAG_NOT_ACTION};
  if (!m) return t;
  const float d = lp - px, e = px - ro;
  if (!isfinite(d) || !isfinite(e) || !isfinite(a)) {
    t.flag = SAO_FLAG_NONFINITE;
    c.nonfin++;
    return t;
  }
  const float w = expf(e);
  if (w <= A.wlo) {
    t.flag = SAO_FLAG_MISMATCH_LOW;
    c.wlow++;
    return t;
  }
  if (w >= A.whi) {
    t.flag = SAO_FLAG_MISMATCH_HIGH;
    c.whigh++;
    return t;
  }
  const float r = expf(d);
  if (a > 0.f && r > A.hi) {
    t.flag = SAO_FLAG_HIGH;
    c.high++;
    contrib += w * (A.hi * a);
  } else if (a < 0.f && r < A.lo) {
    t.flag = SAO_FLAG_LOW;
    c.low++;
    contrib += w * (A.lo * a);
  } else {
    const float v = w * (r * a);
    contrib += v;
    t.flag = SAO_FLAG_IN;
    t.coef = -v * inv_n;
  }
  return t;
}

template <bool kBwd>
__global__ void __launch_bounds__(kThreads) decoupled_loss_kernel(DLArgs a) {
  int64_t n = a.n_norm;
  if (n <= 0) n = total_of(a.cnt_partial, a.n_cnt);
  const float inv_n = n > 0 ? float(1.0 / double(n)) : 0.f;
  const float gscale = kBwd ? __ldg(a.grad_scale) : 1.f;
  double acc = 0.0;
  DLCounts c;
  int n_act = 0;
  const int64_t tid = int64_t(blockIdx.x) * kThreads + threadIdx.x;
  const int64_t stride = int64_t(gridDim.x) * kThreads;
  const bool vec = aligned16_dev(a.logp) && aligned16_dev(a.prox) && aligned16_dev(a.roll) &&
                   aligned16_dev(a.adv) && ((reinterpret_cast<uintptr_t>(a.m) & 3u) == 0) &&
                   (a.coef == nullptr || aligned16_dev(a.coef)) &&
                   (a.flags == nullptr || (reinterpret_cast<uintptr_t>(a.flags) & 3u) == 0);
  int64_t done = 0;
  if (vec) {
    const int64_t n4 = a.N / 4;
    for (int64_t i = tid; i < n4; i += stride) {
      const float4 lp = __ldcs(reinterpret_cast<const float4 *>(a.logp) + i);
      const float4 px = __ldcs(reinterpret_cast<const float4 *>(a.prox) + i);
      const float4 ro = __ldcs(reinterpret_cast<const float4 *>(a.roll) + i);
      const float4 ad = __ldcs(reinterpret_cast<const float4 *>(a.adv) + i);
      const uchar4 mk = __ldcs(reinterpret_cast<const uchar4 *>(a.m) + i);
      if (!kBwd) n_act += nonzero4(mk);
      float contrib = 0.f;
      const PLToken t0 = dl_token(lp.x, px.x, ro.x, ad.x, mk.x, a, inv_n, contrib, c);
      const PLToken t1 = dl_token(lp.y, px.y, ro.y, ad.y, mk.y, a, inv_n, contrib, c);
      const PLToken t2 = dl_token(lp.z, px.z, ro.z, ad.z, mk.z, a, inv_n, contrib, c);
      const PLToken t3 = dl_token(lp.w, px.w, ro.w, ad.w, mk.w, a, inv_n, contrib, c);
      acc += double(contrib);
      if (a.coef)
        __stcs(reinterpret_cast<float4 *>(a.coef) + i,
               make_float4(t0.coef * gscale, t1.coef * gscale, t2.coef * gscale, t3.coef * gscale));
      if (a.flags) reinterpret_cast<uchar4 *>(a.flags)[i] = make_uchar4(t0.flag, t1.flag, t2.flag, t3.flag);
    }
    done = n4 * 4;
  }
  for (int64_t i = done + tid; i < a.N; i += stride) {
    float contrib = 0.f;
    const uint8_t mi = __ldg(a.m + i);
    if (!kBwd) n_act += mi != 0;
    const PLToken t = dl_token(__ldg(a.logp + i), __ldg(a.prox + i), __ldg(a.roll + i), __ldg(a.adv + i),
                               mi, a, inv_n, contrib, c);
    acc += double(contrib);
    if (a.coef) a.coef[i] = t.coef * gscale;
    if (a.flags) a.flags[i] = t.flag;
  }
  if (kBwd) return;
  acc = block_sum(acc);
  const long long k0 = block_sum((long long)c.low), k1 = block_sum((long long)c.high);
  const long long k2 = block_sum((long long)c.nonfin), k3 = block_sum((long long)c.wlow);
  const long long k4 = block_sum((long long)c.whigh);
  const long long na = a.act_out ? block_sum((long long)n_act) : 0;
  if (threadIdx.x == 0) {
    const int g = gridDim.x, b = blockIdx.x;
    if (a.act_out) a.act_out[b] = na;
    a.loss_partial[b] = acc;
    a.cnt5_partial[b] = k0;
    a.cnt5_partial[g + b] = k1;
    a.cnt5_partial[2 * g + b] = k2;
    a.cnt5_partial[3 * g + b] = k3;
    a.cnt5_partial[4 * g + b] = k4;
  }
}

__global__ void __launch_bounds__(kThreads) decoupled_loss_finalize(const double *loss_partial,
                                                                    const long long *cnt5_partial, int grid,
                                                                    const long long *cnt_partial, int n_cnt,
                                                                    int64_t n_norm, float *loss, int64_t *counts) {
  const long long n_action = total_of(cnt_partial, n_cnt);
  double s = 0.0;
  long long k[5] = {0, 0, 0, 0, 0};
  for (int i = threadIdx.x; i < grid; i += kThreads) {
    s += loss_partial[i];
#pragma unroll
    for (int j = 0; j < 5; ++j) k[j] += cnt5_partial[j * grid + i];
  }
  s = block_sum(s);
#pragma unroll
  for (int j = 0; j < 5; ++j) k[j] = block_sum(k[j]);
  if (threadIdx.x == 0) {
    const long long n = n_norm > 0 ? n_norm : n_action;
    *loss = n > 0 ? float(-s / double(n)) : 0.f;
    counts[0] = n_action;
#pragma unroll
    for (int j = 0; j < 5; ++j) counts[1 + j] = k[j];
  }
}

// ---------------------------------------------------------------------------
// value loss
// ---------------------------------------------------------------------------
// Compensated fp32 accumulator (Knuth two-sum): sums millions of terms with
// about twice fp32 precision without fp64 adds in the streaming loop.
struct Acc2 {
  float hi = 0.f, lo = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float s = __fadd_rn(hi, x);
    const float bb = __fsub_rn(s, hi);
    lo = __fadd_rn(lo, __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bb)), __fsub_rn(x, bb)));
    hi = s;
  }
  __device__ __forceinline__ double value() const { return double(hi) + double(lo); }
};

struct VLArgs {
  const float *v, *ret;
  const uint8_t *m;
  int64_t N;
  int64_t n_norm;
  const long long *cnt_partial;
  int n_cnt;
  float *grad;
  double *sums;  // [5][grid]: sum d^2, sum e, sum e^2, sum R, sum R^2
};

// Per-token terms of the value loss and the EV sums, exact up to the final
// additions: d = V - R as an fp32 pair (two-sum), its square and R^2 as a
// rounded product plus the product's remainder (fused multiply-add), so the
// sums are fp64-grade although every operation is fp32.
struct VLTerms {
  Acc2 d2, e, r, r2;  // sum d^2 (= sum (R - V)^2), sum (R - V), sum R, sum R^2: leading parts
  float d2_lo = 0.f, e_lo = 0.f, r2_lo = 0.f;  // their small remainders, summed plainly
  __device__ __forceinline__ void add(float v, float rt) {
    const float dh = __fsub_rn(v, rt);
    const float bb = __fsub_rn(dh, v);
    const float dl = __fsub_rn(__fsub_rn(v, __fsub_rn(dh, bb)), __fadd_rn(rt, bb));  // v - rt = dh + dl exactly
    const float p = __fmul_rn(dh, dh);
    d2.add(p);
    d2_lo = __fadd_rn(d2_lo, __fmaf_rn(2.f * dh, dl, __fmaf_rn(dh, dh, -p)));
    e.add(-dh);
    e_lo = __fsub_rn(e_lo, dl);
    r.add(rt);
    const float q = __fmul_rn(rt, rt);
    r2.add(q);
    r2_lo = __fadd_rn(r2_lo, __fmaf_rn(rt, rt, -q));
  }
};

__global__ void __launch_bounds__(kThreads) value_loss_kernel(VLArgs a) {
  const long long n = a.n_norm > 0 ? a.n_norm : total_of(a.cnt_partial, a.n_cnt);
  const float two_over_n = n > 0 ? float(2.0 / double(n)) : 0.f;
  VLTerms acc;
  const int64_t tid = int64_t(blockIdx.x) * kThreads + threadIdx.x;
  const int64_t stride = int64_t(gridDim.x) * kThreads;
  const bool vec = aligned16_dev(a.v) && aligned16_dev(a.ret) && aligned16_dev(a.grad) &&
                   ((reinterpret_cast<uintptr_t>(a.m) & 3u) == 0);
  auto one = [&](float v, float r, uint8_t m) {
    if (!m) return 0.f;
    acc.add(v, r);
    return two_over_n * (v - r);
  };
  int64_t done = 0;
  if (vec) {
    const int64_t n4 = a.N / 4;
    for (int64_t i = tid; i < n4; i += stride) {
      const float4 v = __ldg(reinterpret_cast<const float4 *>(a.v) + i);
      const float4 r = __ldg(reinterpret_cast<const float4 *>(a.ret) + i);
      const uchar4 m = __ldg(reinterpret_cast<const uchar4 *>(a.m) + i);
      float4 g;
      g.x = one(v.x, r.x, m.x);
      g.y = one(v.y, r.y, m.y);
      g.z = one(v.z, r.z, m.z);
      g.w = one(v.w, r.w, m.w);
      reinterpret_cast<float4 *>(a.grad)[i] = g;
    }
    done = n4 * 4;
  }
  for (int64_t i = done + tid; i < a.N; i += stride)
    a.grad[i] = one(__ldg(a.v + i), __ldg(a.ret + i), __ldg(a.m + i));
  double s_d2 = acc.d2.value() + double(acc.d2_lo), s_e = acc.e.value() + double(acc.e_lo);
  double s_r = acc.r.value(), s_r2 = acc.r2.value() + double(acc.r2_lo);
  s_d2 = block_sum(s_d2);
  s_e = block_sum(s_e);
  s_r = block_sum(s_r);
  s_r2 = block_sum(s_r2);
  if (threadIdx.x == 0) {
    const int g = gridDim.x, b = blockIdx.x;
    a.sums[b] = s_d2;
    a.sums[g + b] = s_e;
    a.sums[2 * g + b] = s_d2;  // sum (R - V)^2 = sum d^2
    a.sums[3 * g + b] = s_r;
    a.sums[4 * g + b] = s_r2;
  }
}

__global__ void __launch_bounds__(kThreads) value_loss_finalize(const double *sums, int grid,
                                                                const long long *cnt_partial, int n_cnt,
                                                                int64_t n_norm, float *loss, double *ev) {
  const long long n = n_norm > 0 ? n_norm : total_of(cnt_partial, n_cnt);
  double s[5] = {0, 0, 0, 0, 0};
  for (int i = threadIdx.x; i < grid; i += kThreads)
#pragma unroll
    for (int k = 0; k < 5; ++k) s[k] += sums[k * grid + i];
#pragma unroll
  for (int k = 0; k < 5; ++k) s[k] = block_sum(s[k]);
  if (threadIdx.x == 0) {
    if (loss) *loss = n > 0 ? float(s[0] / double(n)) : 0.f;
    if (ev) {
      ev[0] = s[1];
      ev[1] = s[2];
      ev[2] = s[3];
      ev[3] = s[4];
    }
  }
}

constexpr int kMaxGrid = 4096;

// Grid of a streaming kernel: one full wave of resident CTAs on this device,
// never more CTAs than 4-token vectors, at most kMaxGrid (workspace bound).
template <class K>
int stream_grid(int64_t N, K kernel) {
  DeviceInfo di;
  int per_sm = 1;
  if (device_info(&di) != SAO_OK) di.sm_count = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, 0) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int64_t want = (N / 4 + kThreads - 1) / kThreads;
  int64_t g = want < 1 ? 1 : want;
  int64_t cap = int64_t(di.sm_count) * per_sm;
  if (cap > kMaxGrid) cap = kMaxGrid;
  return int(g < cap ? g : cap);
}

}  // namespace

// ---------------------------------------------------------------------------
// host launchers
// ---------------------------------------------------------------------------
size_t elementwise_ws_bytes(int64_t N, int) {
  (void)N;
  const int g = kMaxGrid;
  return round256(sizeof(long long) * g) + round256(sizeof(double) * g) +
         round256(3 * sizeof(long long) * g) + round256(5 * sizeof(double) * g);
}

static sao_status launch_count(const uint8_t *m, int64_t N, long long *partial, int grid, cudaStream_t s) {
  int slot = launch_begin("count_mask", s);
  count_mask_kernel<<<grid, kThreads, 0, s>>>(m, N, partial);
  return launch_end(slot, s);
}

sao_status policy_loss_launch(const float *logp, const float *old, const float *adv, const uint8_t *m,
                              int64_t N, float eps_low, float eps_high, int64_t n_norm, float *loss,
                              float *coef, uint8_t *flags, int64_t *counts, const float *grad_loss,
                              void *ws_body, size_t body_bytes, cudaStream_t s) {
  const int grid = grad_loss ? stream_grid(N, policy_loss_kernel<true>) : stream_grid(N, policy_loss_kernel<false>);
  Carver c(ws_body, body_bytes);
  long long *cnt = c.take<long long>(grid);
  double *lossp = c.take<double>(grid);
  long long *cnt3 = c.take<long long>(3 * size_t(grid));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the policy loss");
  // the normaliser must be known before the token pass; with n_norm given,
  // the forward counts the action tokens for `counts` itself
  const bool need_count = n_norm <= 0;
  if (need_count) SAO_TRY(launch_count(m, N, cnt, grid, s));
  PLArgs a;
  a.logp = logp;
  a.old = old;
  a.adv = adv;
  a.m = m;
  a.N = N;
  a.lo = 1.0f - eps_low;
  a.hi = 1.0f + eps_high;
  a.n_norm = n_norm;
  a.cnt_partial = cnt;
  a.n_cnt = need_count ? grid : 0;
  a.act_out = (!need_count && grad_loss == nullptr) ? cnt : nullptr;
  a.coef = coef;
  a.flags = flags;
  a.grad_scale = grad_loss;
  a.loss_partial = lossp;
  a.cnt3_partial = cnt3;
  if (grad_loss) {
    int slot = launch_begin("policy_loss_bwd", s);
    policy_loss_kernel<true><<<grid, kThreads, 0, s>>>(a);
    return launch_end(slot, s);
  }
  int slot = launch_begin("policy_loss_fwd", s);
  policy_loss_kernel<false><<<grid, kThreads, 0, s>>>(a);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("policy_loss_finalize", s);
  policy_loss_finalize<<<1, kThreads, 0, s>>>(lossp, cnt3, grid, cnt, grid, n_norm, loss, counts);
  return launch_end(slot, s);
}

sao_status decoupled_loss_launch(const float *logp, const float *prox, const float *roll, const float *adv,
                                 const uint8_t *m, int64_t N, float eps_low, float eps_high, float w_low,
                                 float w_high, int64_t n_norm, float *loss, float *coef, uint8_t *flags,
                                 int64_t *counts, const float *grad_loss, void *ws_body, size_t body_bytes,
                                 cudaStream_t s) {
  const int grid =
      grad_loss ? stream_grid(N, decoupled_loss_kernel<true>) : stream_grid(N, decoupled_loss_kernel<false>);
  Carver c(ws_body, body_bytes);
  long long *cnt = c.take<long long>(grid);
  double *lossp = c.take<double>(grid);
  long long *cnt5 = c.take<long long>(5 * size_t(grid));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the decoupled loss");
  const bool need_count = n_norm <= 0;
  if (need_count) SAO_TRY(launch_count(m, N, cnt, grid, s));
  DLArgs a;
  a.logp = logp;
  a.prox = prox;
  a.roll = roll;
  a.adv = adv;
  a.m = m;
  a.N = N;
  a.lo = 1.0f - eps_low;
  a.hi = 1.0f + eps_high;
  a.wlo = w_low;
  a.whi = w_high;
  a.n_norm = n_norm;
  a.cnt_partial = cnt;
  a.n_cnt = need_count ? grid : 0;
  a.act_out = (!need_count && grad_loss == nullptr) ? cnt : nullptr;
  a.coef = coef;
  a.flags = flags;
  a.grad_scale = grad_loss;
  a.loss_partial = lossp;
  a.cnt5_partial = cnt5;
  if (grad_loss) {
    int slot = launch_begin("decoupled_loss_bwd", s);
    decoupled_loss_kernel<true><<<grid, kThreads, 0, s>>>(a);
    return launch_end(slot, s);
  }
  int slot = launch_begin("decoupled_loss_fwd", s);
  decoupled_loss_kernel<false><<<grid, kThreads, 0, s>>>(a);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("decoupled_loss_finalize", s);
  decoupled_loss_finalize<<<1, kThreads, 0, s>>>(lossp, cnt5, grid, cnt, grid, n_norm, loss, counts);
  return launch_end(slot, s);
}

sao_status value_loss_launch(const float *v, const float *ret, const uint8_t *m, int64_t N, int64_t n_norm,
                             float *loss, float *grad, double *ev, void *ws_body, size_t body_bytes,
                             cudaStream_t s) {
  const int grid = stream_grid(N, value_loss_kernel);
  Carver c(ws_body, body_bytes);
  long long *cnt = c.take<long long>(grid);
  double *sums = c.take<double>(5 * size_t(grid));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the value loss");
  const bool need_count = n_norm <= 0;  // the normaliser must be known before the token pass
  if (need_count) SAO_TRY(launch_count(m, N, cnt, grid, s));
  VLArgs a{v, ret, m, N, n_norm, cnt, need_count ? grid : 0, grad, sums};
  int slot = launch_begin("value_loss", s);
  value_loss_kernel<<<grid, kThreads, 0, s>>>(a);
  SAO_TRY(launch_end(slot, s));
  slot = launch_begin("value_loss_finalize", s);
  value_loss_finalize<<<1, kThreads, 0, s>>>(sums, grid, cnt, need_count ? grid : 0, n_norm, loss, ev);
  return launch_end(slot, s);
}

}  // namespace sao
