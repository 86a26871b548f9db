// Skip-observation token-level GAE (Preliminaries; §3.2 Eq. 4-5; §4.1) as a
// single-pass reverse scan over packed trajectories.
//
// Formulation. Over the action tokens of one trajectory (observation tokens
// are skipped, Eq. 4-5) write B_j = A_j + V_j, the lambda-return. The GAE
// recursion A_j = r_j + gamma V_{j+1} - V_j + a A_{j+1} (a = gamma lambda)
// becomes
//     B_j = a B_{j+1} + (gamma - a) V_{j+1} + r_j ,   A_j = B_j - V_j ,
// with B = V = 0 after the last action token and r_j = R only on it. The
// return of the critic (lambda_critic) is the same recursion's B itself. This
// form keeps every intermediate O(1) and lets A come out of one final
// subtraction. All of it runs in double-float arithmetic (an fp32 pair, ~48
// significant bits) so long trajectories do not accumulate fp32 rounding.
//
// The state carried right-to-left is S = (B_p, B_c, Vn, P): the two
// lambda-returns of the next action token, its value, and the reward still
// waiting for its action token. Each action token maps S affinely
// (B' = a B + g Vn + P, Vn' = V, P' = 0); the last token of a trajectory
// resets S to (0, 0, 0, R_b). Maps compose associatively, so:
//   * each thread folds its 32 tokens into one map,
//   * a warp-shuffle suffix scan combines the 32 maps of a warp's 1024-token
//     chunk,
//   * warps chain their chunks right-to-left by decoupled look-back: each
//     warp takes a ticket and works on chunk nchunks-1-ticket, so it only
//     ever waits on chunks whose warps started before it; no CTA-wide barrier
//     exists, so a waiting warp never holds up the others; the look-back
//     inspects 32 predecessors at once and composes their maps in log depth;
//     every wait is bounded and a time-out raises SAO_DEVERR_SCAN_TIMEOUT,
//   * each thread then replays its tokens from its incoming state.
// Traffic: values 4 B + mask 1 B read, adv 4 B + ret 4 B written per token.
#include <stdint.h>

#include "sao_common.cuh"
#include "sao_internal.h"
#include "segments.cuh"

namespace sao {
namespace {

constexpr int kThreads = 128;
constexpr int kItems = seg::kItems;       // tokens per lane (at most 32: one bit each)
constexpr int kChunk = seg::kSegChunk;    // tokens per warp chunk
constexpr int kWarps = kThreads / 32;

// ---------------------------------------------------------------------------
// double-float arithmetic (Dekker / Knuth error-free transformations)
// ---------------------------------------------------------------------------
struct df {
  float hi, lo;
};
__device__ __forceinline__ df quick_two_sum(float a, float b) {  // |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ df two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
__device__ __forceinline__ df df_add(df x, df y) {
  const df s = two_sum(x.hi, y.hi);
  return quick_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(x.lo, y.lo)));
}
__device__ __forceinline__ df df_add_f(df x, float y) {
  const df s = two_sum(x.hi, y);
  return quick_two_sum(s.hi, __fadd_rn(s.lo, x.lo));
}
__device__ __forceinline__ df df_mul(df x, df y) {
  const float p = __fmul_rn(x.hi, y.hi);
  float e = __fmaf_rn(x.hi, y.hi, -p);
  e = __fmaf_rn(x.hi, y.lo, e);
  e = __fmaf_rn(x.lo, y.hi, e);
  return quick_two_sum(p, e);
}
__device__ __forceinline__ df df_mul_f(df x, float y) {
  const float p = __fmul_rn(x.hi, y);
  float e = __fmaf_rn(x.hi, y, -p);
  e = __fmaf_rn(x.lo, y, e);
  return quick_two_sum(p, e);
}
__device__ __forceinline__ float df_round(df x) { return __fadd_rn(x.hi, x.lo); }
__device__ __forceinline__ df df_from_double(double x) {
  const float hi = float(x);
  return {hi, float(x - double(hi))};
}

// Per-trajectory coefficients: a = gamma*lambda and g = gamma - a for the
// policy (lambda_b) and the critic (lambda_critic).
struct TCoef {
  df ap, gp, ac, gc;
};
__device__ __forceinline__ TCoef load_coef(const float4 *tab, int b) {
  const float4 u = __ldg(tab + 2 * b), w = __ldg(tab + 2 * b + 1);
  return {{u.x, u.y}, {u.z, u.w}, {w.x, w.y}, {w.z, w.w}};
}

// The affine map of a token segment, from the state at its right edge to the
// state at its left edge. fl bit 0: the segment holds the last token of a
// trajectory (the map ignores the incoming state); bit 1: the segment (left of
// any reset) holds an action token. Identity when fl == 0.
//   reset:          B = c,                        Vn = act ? v : 0, P = act ? 0 : p0
//   act, no reset:  B = ap (a B + g Vn + P) + c,  Vn = v,           P = 0
// b is the trajectory of the segment's leftmost token.
struct GMap {
  int b, fl;
  df ap, cp, ac, cc;
  float v, p0;
  TCoef k;  // coefficients of trajectory b (used when the map is the left operand)
};
struct GState {
  df Bp, Bc;
  float Vn, P;
};

__device__ __forceinline__ GMap identity_map() {
  GMap m;
  m.b = 0;
  m.fl = 0;
  m.ap = m.ac = {1.f, 0.f};
  m.cp = m.cc = {0.f, 0.f};
  m.v = m.p0 = 0.f;
  m.k = TCoef{};
  return m;
}

// x o y: x is the left segment, y the one immediately to its right.
template <bool kCrit>
__device__ GMap compose(const GMap &x, const GMap &y, const float4 *) {
  if (x.fl & 1) return x;
  if (!(x.fl & 2)) return y;
  if (!(y.fl & 3)) return x;
  const TCoef &c = x.k;
  const bool yact = (y.fl & 2) != 0;
  const float Yv = yact ? y.v : 0.f, Yp = yact ? 0.f : y.p0;
  GMap r;
  r.b = x.b;
  r.k = x.k;
  r.v = x.v;
  r.p0 = 0.f;
  df tp = df_add_f(df_add(df_mul(c.ap, y.cp), df_mul_f(c.gp, Yv)), Yp);
  r.cp = df_add(df_mul(x.ap, tp), x.cp);
  if (kCrit) {
    df tc = df_add_f(df_add(df_mul(c.ac, y.cc), df_mul_f(c.gc, Yv)), Yp);
    r.cc = df_add(df_mul(x.ac, tc), x.cc);
  } else {
    r.cc = {0.f, 0.f};
  }
  if (y.fl & 1) {
    r.fl = 3;
    r.ap = r.ac = {0.f, 0.f};
  } else {
    r.fl = 2;
    r.ap = df_mul(df_mul(x.ap, c.ap), y.ap);
    r.ac = kCrit ? df_mul(df_mul(x.ac, c.ac), y.ac) : df{1.f, 0.f};
  }
  return r;
}

template <bool kCrit>
__device__ GState apply(const GMap &m, const GState &s, const float4 *) {
  if (m.fl & 1) {
    const bool act = (m.fl & 2) != 0;
    return {m.cp, m.cc, act ? m.v : 0.f, act ? 0.f : m.p0};
  }
  if (!(m.fl & 2)) return s;
  const TCoef &c = m.k;
  GState r;
  const df tp = df_add_f(df_add(df_mul(c.ap, s.Bp), df_mul_f(c.gp, s.Vn)), s.P);
  r.Bp = df_add(df_mul(m.ap, tp), m.cp);
  if (kCrit) {
    const df tc = df_add_f(df_add(df_mul(c.ac, s.Bc), df_mul_f(c.gc, s.Vn)), s.P);
    r.Bc = df_add(df_mul(m.ac, tc), m.cc);
  } else {
    r.Bc = {0.f, 0.f};
  }
  r.Vn = m.v;
  r.P = 0.f;
  return r;
}

__device__ __forceinline__ GMap shfl_down_map(const GMap &m, int d) {
  GMap r;
  r.b = __shfl_down_sync(0xffffffffu, m.b, d);
  r.fl = __shfl_down_sync(0xffffffffu, m.fl, d);
  r.ap.hi = __shfl_down_sync(0xffffffffu, m.ap.hi, d);
  r.ap.lo = __shfl_down_sync(0xffffffffu, m.ap.lo, d);
  r.cp.hi = __shfl_down_sync(0xffffffffu, m.cp.hi, d);
  r.cp.lo = __shfl_down_sync(0xffffffffu, m.cp.lo, d);
  r.ac.hi = __shfl_down_sync(0xffffffffu, m.ac.hi, d);
  r.ac.lo = __shfl_down_sync(0xffffffffu, m.ac.lo, d);
  r.cc.hi = __shfl_down_sync(0xffffffffu, m.cc.hi, d);
  r.cc.lo = __shfl_down_sync(0xffffffffu, m.cc.lo, d);
  r.v = __shfl_down_sync(0xffffffffu, m.v, d);
  r.p0 = __shfl_down_sync(0xffffffffu, m.p0, d);
  r.k.ap.hi = __shfl_down_sync(0xffffffffu, m.k.ap.hi, d);
  r.k.ap.lo = __shfl_down_sync(0xffffffffu, m.k.ap.lo, d);
  r.k.gp.hi = __shfl_down_sync(0xffffffffu, m.k.gp.hi, d);
  r.k.gp.lo = __shfl_down_sync(0xffffffffu, m.k.gp.lo, d);
  r.k.ac.hi = __shfl_down_sync(0xffffffffu, m.k.ac.hi, d);
  r.k.ac.lo = __shfl_down_sync(0xffffffffu, m.k.ac.lo, d);
  r.k.gc.hi = __shfl_down_sync(0xffffffffu, m.k.gc.hi, d);
  r.k.gc.lo = __shfl_down_sync(0xffffffffu, m.k.gc.lo, d);
  return r;
}

// ---------------------------------------------------------------------------
// cross-CTA publication (decoupled look-back)
// ---------------------------------------------------------------------------
struct __align__(16) ChunkPub {
  GMap agg;     // map of the whole chunk (status >= 1)
  GState incl;  // state at the chunk's left edge (status == 2)
};

__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int *p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Published maps and states go through L2 only (st.cg / ld.cg), so a reader on
// another SM never sees a stale L1 line.
__device__ __forceinline__ void st_df(df *p, df x) {
  __stcg(&p->hi, x.hi);
  __stcg(&p->lo, x.lo);
}
__device__ __forceinline__ df ld_df(const df *p) { return {__ldcg(&p->hi), __ldcg(&p->lo)}; }
__device__ void store_map(GMap *p, const GMap &m) {
  __stcg(&p->b, m.b);
  __stcg(&p->fl, m.fl);
  st_df(&p->ap, m.ap);
  st_df(&p->cp, m.cp);
  st_df(&p->ac, m.ac);
  st_df(&p->cc, m.cc);
  __stcg(&p->v, m.v);
  __stcg(&p->p0, m.p0);
  st_df(&p->k.ap, m.k.ap);
  st_df(&p->k.gp, m.k.gp);
  st_df(&p->k.ac, m.k.ac);
  st_df(&p->k.gc, m.k.gc);
}
__device__ GMap load_map(const GMap *p) {
  GMap m;
  m.b = __ldcg(&p->b);
  m.fl = __ldcg(&p->fl);
  m.ap = ld_df(&p->ap);
  m.cp = ld_df(&p->cp);
  m.ac = ld_df(&p->ac);
  m.cc = ld_df(&p->cc);
  m.v = __ldcg(&p->v);
  m.p0 = __ldcg(&p->p0);
  m.k.ap = ld_df(&p->k.ap);
  m.k.gp = ld_df(&p->k.gp);
  m.k.ac = ld_df(&p->k.ac);
  m.k.gc = ld_df(&p->k.gc);
  return m;
}
__device__ void store_state(GState *p, const GState &s) {
  st_df(&p->Bp, s.Bp);
  st_df(&p->Bc, s.Bc);
  __stcg(&p->Vn, s.Vn);
  __stcg(&p->P, s.P);
}
__device__ GState load_state(const GState *p) {
  GState s;
  s.Bp = ld_df(&p->Bp);
  s.Bc = ld_df(&p->Bc);
  s.Vn = __ldcg(&p->Vn);
  s.P = __ldcg(&p->P);
  return s;
}

// Waits until *p != 0; returns it, or 0 after kWaitLimitNs / kSpinLimit polls.
__device__ int wait_nonzero(const int *p) {
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t n = 0; n < kSpinLimit; ++n) {
    const int s = ld_acquire(p);
    if (s != 0) return s;
    if ((n & 63u) == 63u && globaltimer_ns() - t0 > kWaitLimitNs) return 0;
    __nanosleep(64);
  }
  return 0;
}

struct GaeArgs {
  const float *values, *rewards;
  const uint8_t *m;
  const int32_t *cu;
  int B;
  int64_t N;
  int nchunks;
  const float4 *coef;  // [B][2]
  const int *chunk_first;  // [nchunks] trajectory of each chunk's first token
  int *ticket;
  int *status;         // [nchunks]
  ChunkPub *pub;       // [nchunks]
  float *adv, *ret;
  unsigned int *err;
};

using seg::CuView;
using seg::find_traj;
using seg::kCuCap;

// State at the right edge of chunk q, from the chunks to its right. The warp
// inspects 32 successors (q+1 .. q+32) per round: each lane polls one status
// word; the first chunk whose left-edge state is known (published inclusive
// state, a map that ignores its right neighbour, or the end of the input) ends
// the walk, and the maps of the chunks before it are composed by a log-depth
// shuffle scan. A round waits (bounded) only for chunks before that point.
template <bool kCrit>
__device__ GState look_back(const GaeArgs &a, int q, int lane) {
  GState zero;
  zero.Bp = zero.Bc = {0.f, 0.f};
  zero.Vn = zero.P = 0.f;
  GMap acc = identity_map();  // maps of the chunks already walked (lane 0)
  const uint64_t t_start = globaltimer_ns();
  for (int base = q + 1;; base += 32) {
    const int j = base + lane;
    int st = 0;
    GMap mj = identity_map();
    bool term = false;
    uint32_t polls = 0;
    for (;;) {
      st = j < a.nchunks ? ld_acquire(a.status + j) : 2;
      term = (st == 2);
      if (st == 1) {
        mj = load_map(&a.pub[j].agg);
        term = (mj.fl & 1) != 0;
      }
      const unsigned bt = __ballot_sync(0xffffffffu, term);
      const unsigned bn = __ballot_sync(0xffffffffu, st == 0);
      const int first_term = bt ? __ffs(bt) - 1 : 32;
      const int first_nr = bn ? __ffs(bn) - 1 : 32;
      if (first_nr >= first_term) break;  // everything up to the first terminal chunk is known
      if ((++polls & 31u) == 0u && globaltimer_ns() - t_start > kWaitLimitNs) {
        if (lane == 0) raise_device_error(a.err, SAO_DEVERR_SCAN_TIMEOUT);
        return zero;
      }
      __nanosleep(128);
    }
    const unsigned bt = __ballot_sync(0xffffffffu, term);
    const int stop = bt ? __ffs(bt) - 1 : 32;
    // state at the left edge of the terminal chunk (if any in this round)
    GState tstate = zero;
    if (lane == stop && j < a.nchunks) tstate = (st == 2) ? load_state(&a.pub[j].incl) : apply<kCrit>(mj, zero, a.coef);
    // compose maps of lanes [0, stop): suffix scan, lane 0 ends with m_0 o ... o m_{stop-1}
    GMap m = lane < stop ? mj : identity_map();
#pragma unroll 1
    for (int d = 1; d < 32; d <<= 1) {
      const GMap o = shfl_down_map(m, d);
      if (lane + d < 32) m = compose<kCrit>(m, o, a.coef);
    }
    if (lane == 0) acc = compose<kCrit>(acc, m, a.coef);
    if (stop < 32) {
      tstate.Bp.hi = __shfl_sync(0xffffffffu, tstate.Bp.hi, stop);
      tstate.Bp.lo = __shfl_sync(0xffffffffu, tstate.Bp.lo, stop);
      tstate.Bc.hi = __shfl_sync(0xffffffffu, tstate.Bc.hi, stop);
      tstate.Bc.lo = __shfl_sync(0xffffffffu, tstate.Bc.lo, stop);
      tstate.Vn = __shfl_sync(0xffffffffu, tstate.Vn, stop);
      tstate.P = __shfl_sync(0xffffffffu, tstate.P, stop);
      GState r = apply<kCrit>(acc, tstate, a.coef);  // meaningful in lane 0
      r.Bp.hi = __shfl_sync(0xffffffffu, r.Bp.hi, 0);
      r.Bp.lo = __shfl_sync(0xffffffffu, r.Bp.lo, 0);
      r.Bc.hi = __shfl_sync(0xffffffffu, r.Bc.hi, 0);
      r.Bc.lo = __shfl_sync(0xffffffffu, r.Bc.lo, 0);
      r.Vn = __shfl_sync(0xffffffffu, r.Vn, 0);
      r.P = __shfl_sync(0xffffffffu, r.P, 0);
      return r;
    }
  }
}

// Per-warp staging of a 1024-token chunk in shared memory: global memory is
// read and written with fully coalesced 16-byte accesses, while each lane
// works on its own run of 32 consecutive tokens. Rows are padded (33 floats,
// 36 bytes) so lane-major reads hit 32 different banks.
constexpr int kPadF = kItems + 1;
constexpr int kPadB = kItems + 4;
struct WarpStage {
  float val[32][kPadF];   // values in, advantages out
  float ret[32][kPadF];   // returns out
  uint8_t msk[32][kPadB]; // action flags
};

__device__ __forceinline__ void stage_in(const GaeArgs &a, int64_t c0, int lane, WarpStage &ws) {
  const int64_t N = a.N;
  const bool full = c0 + kChunk <= N && aligned16_dev(a.values) && aligned16_dev(a.m);
  if (full) {
#pragma unroll
    for (int it = 0; it < kChunk / 128; ++it) {
      const int i = it * 128 + lane * 4;
      const float4 x = __ldcs(reinterpret_cast<const float4 *>(a.values + c0 + i));
      float *d = &ws.val[i / kItems][i % kItems];
      d[0] = x.x;
      d[1] = x.y;
      d[2] = x.z;
      d[3] = x.w;
    }
#pragma unroll
    for (int it = 0; it < kChunk / 512; ++it) {
      const int i = it * 512 + lane * 16;
      const uint4 x = __ldcs(reinterpret_cast<const uint4 *>(a.m + c0 + i));
      uint32_t *d = reinterpret_cast<uint32_t *>(&ws.msk[i / kItems][i % kItems]);
      d[0] = x.x;
      d[1] = x.y;
      d[2] = x.z;
      d[3] = x.w;
    }
  } else {
    for (int i = lane; i < kChunk; i += 32) {
      const int64_t t = c0 + i;
      ws.val[i / kItems][i % kItems] = t < N ? a.values[t] : 0.f;
      ws.msk[i / kItems][i % kItems] = (t < N && a.m[t] != 0) ? 1 : 0;
    }
  }
  __syncwarp();
}

__device__ __forceinline__ void stage_out(const GaeArgs &a, int64_t c0, int lane, const WarpStage &ws) {
  __syncwarp();
  const int64_t N = a.N;
  const bool full = c0 + kChunk <= N && aligned16_dev(a.adv) && aligned16_dev(a.ret);
  if (full) {
#pragma unroll
    for (int it = 0; it < kChunk / 128; ++it) {
      const int i = it * 128 + lane * 4;
      const float *v = &ws.val[i / kItems][i % kItems];
      const float *r = &ws.ret[i / kItems][i % kItems];
      __stcs(reinterpret_cast<float4 *>(a.adv + c0 + i), make_float4(v[0], v[1], v[2], v[3]));
      __stcs(reinterpret_cast<float4 *>(a.ret + c0 + i), make_float4(r[0], r[1], r[2], r[3]));
    }
  } else {
    for (int i = lane; i < kChunk; i += 32) {
      const int64_t t = c0 + i;
      if (t < N) {
        a.adv[t] = ws.val[i / kItems][i % kItems];
        a.ret[t] = ws.ret[i / kItems][i % kItems];
      }
    }
  }
}

template <bool kCrit>
__global__ void __launch_bounds__(kThreads, 4) gae_scan_kernel(GaeArgs a) {
  __shared__ int32_t s_cu_all[kWarps][kCuCap];
  __shared__ WarpStage s_stage[kWarps];
  __shared__ int s_ticket;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // One ticket per CTA: its warps take consecutive chunks, highest first, so
  // every chunk a warp waits on belongs to a CTA (or a warp) already running.
  if (threadIdx.x == 0) s_ticket = atomicAdd(a.ticket, kWarps);
  __syncthreads();
  const int q = a.nchunks - 1 - (s_ticket + warp);
  if (q < 0) return;  // the grid rounds the warp count up to whole CTAs
  const int64_t t0 = int64_t(q) * kChunk + int64_t(lane) * kItems;
  const int64_t N = a.N;

  // This chunk's slice of cu_seqlens, in shared memory when it fits.
  const int blo = __ldg(a.chunk_first + q);
  const int bhi = q + 1 < a.nchunks ? __ldg(a.chunk_first + q + 1) : a.B - 1;
  const int ncu = bhi - blo + 2;  // cu[blo .. bhi + 1]
  int32_t *s_cu = s_cu_all[warp];
  const CuView cu{a.cu, s_cu, blo, ncu <= kCuCap};
  if (cu.in_smem)
    for (int i = lane; i < ncu; i += 32) s_cu[i] = __ldg(a.cu + blo + i);
  __syncwarp();
  WarpStage &stg = s_stage[warp];
  stage_in(a, int64_t(q) * kChunk, lane, stg);
  const float *vrow = stg.val[lane];
  const uint8_t *mrow = stg.msk[lane];

  // ---- trajectory ends among the 16 tokens (forward walk over cu_seqlens) -------
  uint32_t endbits = 0;
  int b_last;
  {
    int b = cu.find(blo, bhi, t0 < N ? t0 : N - 1);
    int64_t next_end = cu[b + 1];
    bool bad = false;
#pragma unroll 4
    for (int k = 0; k < kItems; ++k) {
      const int64_t t = t0 + k;
      if (t < N) {
        while (b < bhi && t >= next_end) {
          ++b;
          next_end = cu[b + 1];
        }
        bad |= (t >= next_end);  // cu_seqlens[B] < N
        endbits |= uint32_t(t == next_end - 1) << k;
      }
    }
    b_last = b;
    if (bad) raise_device_error(a.err, SAO_DEVERR_CU_SEQLENS);
  }

  // ---- fold the thread's tokens into one map (right to left) ------------------
  GMap M = identity_map();
  {
    int b = b_last;
    int64_t b_start = cu[b];
    TCoef c = load_coef(a.coef, b);
#pragma unroll 1
    for (int g = kItems / 4 - 1; g >= 0; --g) {
      float v[4];
      uint32_t act4 = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[i] = vrow[4 * g + i];
        act4 |= uint32_t(mrow[4 * g + i] != 0) << i;
      }
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        const int k = 4 * g + i;
        const int64_t t = t0 + k;
        if (t < b_start && t < N) {
          while (b > blo && t < b_start) {
            --b;
            b_start = cu[b];
          }
          c = load_coef(a.coef, b);
        }
        const bool is_act = (act4 >> i) & 1u, is_end = (endbits >> k) & 1u;
        if (is_end) {
          const float R = __ldg(a.rewards + b);
          M.b = b;
          M.ap = M.ac = {0.f, 0.f};
          M.fl = is_act ? 3 : 1;
          M.cp = M.cc = {is_act ? R : 0.f, 0.f};
          M.v = is_act ? v[i] : 0.f;
          M.p0 = is_act ? 0.f : R;
        } else if (is_act) {
          if (M.fl == 0) {
            M.fl = 2;
            M.ap = M.ac = {1.f, 0.f};
            M.cp = M.cc = {0.f, 0.f};
          } else {
            const bool mact = (M.fl & 2) != 0;
            const float Yv = mact ? M.v : 0.f, Yp = mact ? 0.f : M.p0;
            M.cp = df_add(df_mul(c.ap, M.cp), df_mul_f(c.gp, Yv));
            if (kCrit) M.cc = df_add(df_mul(c.ac, M.cc), df_mul_f(c.gc, Yv));
            if (Yp != 0.f) {  // only right after a trajectory that ends on observations
              M.cp = df_add_f(M.cp, Yp);
              if (kCrit) M.cc = df_add_f(M.cc, Yp);
            }
            if (!(M.fl & 1)) {
              M.ap = df_mul(c.ap, M.ap);
              if (kCrit) M.ac = df_mul(c.ac, M.ac);
            }
            M.fl |= 2;
          }
          M.b = b;
          M.v = v[i];
          M.p0 = 0.f;
        } else if (M.fl != 0) {
          M.b = b;
        }
      }
    }
    M.k = c;  // M.b, when the map is not the identity, is the trajectory of the leftmost token: b
  }

  // ---- suffix scan of the 32 maps of this warp ------------------------------------
  GMap S = M;
#pragma unroll 1
  for (int d = 1; d < 32; d <<= 1) {
    const GMap o = shfl_down_map(S, d);
    if (lane + d < 32) S = compose<kCrit>(S, o, a.coef);
  }
  GMap E = shfl_down_map(S, 1);  // lanes to my right within the chunk
  if (lane == 31) E = identity_map();

  // ---- publish this chunk and look back for the state at its right edge ------------
  // Release stores of the status word order the published map/state before it;
  // readers acquire the status before reading them.
  GState zero;
  zero.Bp = zero.Bc = {0.f, 0.f};
  zero.Vn = zero.P = 0.f;
  const bool last = (q == a.nchunks - 1);
  const bool reset = (S.fl & 1) != 0;  // lane 0 holds the chunk's map
  ChunkPub *me = a.pub + q;
  if (lane == 0) {
    // A chunk whose map ignores its right neighbour publishes its left-edge
    // state at once; the others publish their map first.
    if (last || reset) {
      store_state(&me->incl, apply<kCrit>(S, zero, a.coef));
      st_release(a.status + q, 2);
    } else {
      store_map(&me->agg, S);
      st_release(a.status + q, 1);
    }
  }
  GState right = zero;
  if (!__shfl_sync(0xffffffffu, int(last), 0)) right = look_back<kCrit>(a, q, lane);
  if (lane == 0 && !reset && !last) {
    store_state(&me->incl, apply<kCrit>(S, right, a.coef));
    st_release(a.status + q, 2);
  }

  // ---- replay the tokens from the incoming state ----------------------------------
  GState st = apply<kCrit>(E, right, a.coef);
  {
    int b = b_last;
    int64_t b_start = cu[b];
    TCoef c = load_coef(a.coef, b);
    float R = __ldg(a.rewards + b);
    float *orow = stg.val[lane];
    float *rrow = stg.ret[lane];
#pragma unroll 1
    for (int g = kItems / 4 - 1; g >= 0; --g) {
      float v[4], ov[4], orr[4];
      uint32_t act4 = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        v[i] = vrow[4 * g + i];
        act4 |= uint32_t(mrow[4 * g + i] != 0) << i;
      }
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        const int k = 4 * g + i;
        const int64_t t = t0 + k;
        ov[i] = 0.f;
        orr[i] = 0.f;
        if (t >= N) continue;
        if (t < b_start) {
          while (b > blo && t < b_start) {
            --b;
            b_start = cu[b];
          }
          c = load_coef(a.coef, b);
          R = __ldg(a.rewards + b);
        }
        if ((endbits >> k) & 1u) {
          st.Bp = st.Bc = {0.f, 0.f};
          st.Vn = 0.f;
          st.P = R;
        }
        if ((act4 >> i) & 1u) {
          st.Bp = df_add(df_mul(c.ap, st.Bp), df_mul_f(c.gp, st.Vn));
          if (kCrit) st.Bc = df_add(df_mul(c.ac, st.Bc), df_mul_f(c.gc, st.Vn));
          if (st.P != 0.f) {
            st.Bp = df_add_f(st.Bp, st.P);
            if (kCrit) st.Bc = df_add_f(st.Bc, st.P);
          }
          orr[i] = kCrit ? df_round(st.Bc) : R;  // gamma = lambda_critic = 1: the return is R
          ov[i] = df_round(df_add_f(st.Bp, -v[i]));
          st.Vn = v[i];
          st.P = 0.f;
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        orow[4 * g + i] = ov[i];
        rrow[4 * g + i] = orr[i];
      }
    }
  }
  stage_out(a, int64_t(q) * kChunk, lane, stg);
}

// Per-trajectory coefficients (fp64 then split to double-float) and a check of
// cu_seqlens: 0 = cu[0] <= cu[1] <= ... <= cu[B] = N.
__global__ void gae_coef_kernel(const int32_t *cu, int B, int64_t N, float gamma, float lam, float lam_c,
                                float alpha, const int *nact, float4 *coef, unsigned int *err) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  if ((b == 0 && cu[0] != 0) || cu[b + 1] < cu[b] || (b == B - 1 && int64_t(cu[B]) != N))
    raise_device_error(err, SAO_DEVERR_CU_SEQLENS);
  double lb = lam;
  if (alpha > 0.f) {
    const int L = nact[b];
    lb = L > 0 ? 1.0 - 1.0 / (double(alpha) * double(L)) : 0.0;
    lb = lb < 0.0 ? 0.0 : (lb > 1.0 ? 1.0 : lb);
  }
  const double g = gamma;
  const double ap = g * lb, ac = g * double(lam_c);
  const df Ap = df_from_double(ap), Gp = df_from_double(g - ap);
  const df Ac = df_from_double(ac), Gc = df_from_double(g - ac);
  coef[2 * b] = make_float4(Ap.hi, Ap.lo, Gp.hi, Gp.lo);
  coef[2 * b + 1] = make_float4(Ac.hi, Ac.lo, Gc.hi, Gc.lo);
}

}  // namespace

size_t gae_ws_bytes(int64_t N, int64_t B) {
  const int64_t nchunks = (N + kChunk - 1) / kChunk;
  return round256(sizeof(int)) + round256(sizeof(int) * (B + 1)) + round256(sizeof(int) * nchunks) +
         round256(sizeof(float4) * 2 * (B + 1)) + round256(sizeof(ChunkPub) * nchunks) +
         round256(sizeof(int) * (nchunks + 1));
}

sao_status gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu,
                      int32_t B, int64_t N, float gamma, float lam, float lam_c, float alpha, float *adv,
                      float *ret, unsigned int *err, void *ws_body, size_t body_bytes, cudaStream_t s) {
  if (N == 0) return SAO_OK;
  const int64_t nchunks = (N + kChunk - 1) / kChunk;
  if (nchunks > (int64_t(1) << 30)) return fail(SAO_ERR_SHAPE, "too many tokens for the advantage scan");
  Carver c(ws_body, body_bytes);
  char *zero_begin = c.base + c.off;
  int *ticket = c.take<int>(1);
  int *nact = c.take<int>(size_t(B) + 1);
  int *status = c.take<int>(size_t(nchunks));
  char *zero_end = c.base + c.off;
  float4 *coef = c.take<float4>(2 * (size_t(B) + 1));
  ChunkPub *pub = c.take<ChunkPub>(size_t(nchunks));
  int *chunk_first = c.take<int>(size_t(nchunks) + 1);
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the advantage scan");
  SAO_CUDA_TRY(cudaMemsetAsync(zero_begin, 0, size_t(zero_end - zero_begin), s));
  {
    int slot = launch_begin("gae_chunk_first", s);
    seg::chunk_first_kernel<<<unsigned((nchunks + 255) / 256), 256, 0, s>>>(cu, B, N, int(nchunks), chunk_first);
    SAO_TRY(launch_end(slot, s));
  }
  if (alpha > 0.f) {
    int slot = launch_begin("gae_count", s);
    seg::action_count_kernel<<<unsigned((nchunks + 7) / 8), 256, 0, s>>>(m, cu, B, N, int(nchunks),
                                                                                    chunk_first, nact);
    SAO_TRY(launch_end(slot, s));
  }
  {
    int slot = launch_begin("gae_coef", s);
    gae_coef_kernel<<<(B + 127) / 128, 128, 0, s>>>(cu, B, N, gamma, lam, lam_c, alpha, nact, coef, err);
    SAO_TRY(launch_end(slot, s));
  }
  GaeArgs a;
  a.values = values;
  a.rewards = rewards;
  a.m = m;
  a.cu = cu;
  a.B = B;
  a.N = N;
  a.nchunks = int(nchunks);
  a.coef = coef;
  a.chunk_first = chunk_first;
  a.ticket = ticket;
  a.status = status;
  a.pub = pub;
  a.adv = adv;
  a.ret = ret;
  a.err = err;
  const bool crit_trivial = (gamma == 1.0f && lam_c == 1.0f);
  const unsigned grid = unsigned((nchunks + kWarps - 1) / kWarps);
  int slot = launch_begin("gae_scan", s);
  if (crit_trivial)
    gae_scan_kernel<false><<<grid, kThreads, 0, s>>>(a);
  else
    gae_scan_kernel<true><<<grid, kThreads, 0, s>>>(a);
  return launch_end(slot, s);
}

}  // namespace sao
