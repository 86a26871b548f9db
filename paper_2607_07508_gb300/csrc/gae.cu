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
// waiting for its action token (P != 0 only in the state a trajectory end
// leaves, where B = Vn = 0). Each action token maps S affinely
// (B' = a B + g Vn + P, Vn' = V, P' = 0); the last token of a trajectory
// resets S to (0, 0, 0, R_b). Maps compose associatively, so:
//   * a warp owns a chunk of 32 lane segments, each lane 32 * pieces
//     consecutive tokens (pieces = 1, 2 or 4, from N); the segments stream
//     through shared memory one 32-token piece at a time, one TMA tensor
//     copy for the values and one for the mask (the arrays seen as a row per
//     lane segment, rows swizzled so that the lane-major row reads are free
//     of bank conflicts), and the results leave the same way,
//   * each lane folds its segment into one map, driven by two bit masks
//     (action tokens; trajectory ends, marked once per chunk from its
//     cu_seqlens slice) so the common token costs one fused double-float
//     a*B + g*V, a few selects and no index arithmetic, and keeps its values
//     in its own TMEM lane for the replay (the scan issues no MMA, so the
//     SM's 256 KB of TMEM is free: 4 CTAs x 128 columns),
//   * a warp-shuffle suffix scan combines the 32 maps of the chunk,
//   * warps chain their chunks right-to-left by decoupled look-back: chunks
//     are taken by ticket, so a warp only ever waits on chunks taken before
//     its own; the look-back polls 32 predecessors at once and carries the
//     nearest known state through the maps before it one by one (so results
//     do not depend on timing); maps and states are published as tagged
//     8-byte words, so neither side needs a fence; every wait is bounded and
//     a time-out raises SAO_DEVERR_SCAN_TIMEOUT,
//   * each lane then replays its tokens from TMEM, starting from its incoming
//     state, writing A and the return into shared memory, from where one
//     tensor store each takes them out.
// Traffic: values 4 B + mask 1 B read, adv 4 B + ret 4 B written per token.
#include <stdint.h>

#include <mutex>

#include "sao_common.cuh"
#include "sao_internal.h"
#include "segments.cuh"
#include "tc_ptx.cuh"

namespace sao {
namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;
constexpr int kMinBlocks = 4;             // 16 warps per SM (shared memory and TMEM bound)
constexpr int kMaxPieces = 4;             // 32-token pieces per lane segment, at most
constexpr int kTmemCols = 32 * kMaxPieces;  // TMEM columns per CTA: 4 CTAs fill an SM's 512
constexpr int kItems = seg::kItems;       // tokens per lane (one bit each)
constexpr int kChunk = seg::kSegChunk;    // tokens per warp chunk
static_assert(kItems == 32 && kChunk == 1024, "the staging layout assumes 32 x 32 tokens per warp");

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
__device__ __forceinline__ df df_mul(df x, df y) {
  const float p = __fmul_rn(x.hi, y.hi);
  float e = __fmaf_rn(x.hi, y.hi, -p);
  e = __fmaf_rn(x.hi, y.lo, e);
  e = __fmaf_rn(x.lo, y.hi, e);
  return quick_two_sum(p, e);
}
// a*x + g*v for double-float a, x, g and a float v: both products split
// exactly (FMA), their high parts added exactly (two-sum), the low-order terms
// gathered in one float and renormalised once. a.lo*x.lo and g.lo*v's
// rounding are below the format's precision.
__device__ __forceinline__ df df_axpby(df a, df x, df g, float v) {
  const float p1 = __fmul_rn(a.hi, x.hi);
  const float e1 = __fmaf_rn(a.hi, x.hi, -p1);
  const float p2 = __fmul_rn(g.hi, v);
  const float e2 = __fmaf_rn(g.hi, v, -p2);
  const df s = two_sum(p1, p2);
  float lo = __fmaf_rn(a.hi, x.lo, e1);
  lo = __fmaf_rn(a.lo, x.hi, lo);
  lo = __fmaf_rn(g.lo, v, lo);
  lo = __fadd_rn(lo, e2);
  lo = __fadd_rn(lo, s.lo);
  return quick_two_sum(s.hi, lo);
}
// The same a*x + g*v with the result left unnormalised: (s, lo), which the
// next step's products take as they are (every term of lo is carried, none
// dropped). Each step adds a few ulps of s to lo, so over the 32 tokens
// between the renormalisations of the branch-free loops (once per piece) lo
// stays within about a hundred ulps of s, and its own fp32 roundings stay
// near 2^-40 of the value.
__device__ __forceinline__ df df_axpby_u(df a, df x, df g, float v) {
  const float p1 = __fmul_rn(a.hi, x.hi);
  const float e1 = __fmaf_rn(a.hi, x.hi, -p1);
  const float p2 = __fmul_rn(g.hi, v);
  const float e2 = __fmaf_rn(g.hi, v, -p2);
  const df s = two_sum(p1, p2);
  float lo = __fmaf_rn(a.hi, x.lo, e1);
  lo = __fmaf_rn(a.lo, x.hi, lo);
  lo = __fmaf_rn(g.lo, v, lo);
  lo = __fadd_rn(lo, e2);
  return {s.hi, __fadd_rn(lo, s.lo)};
}
__device__ __forceinline__ df df_renorm(df x) { return two_sum(x.hi, x.lo); }
// x^e for 0 <= e < 32 by squaring.
__device__ df df_pow(df x, int e) {
  df r = {1.f, 0.f};
#pragma unroll 1
  while (e) {
    if (e & 1) r = df_mul(r, x);
    e >>= 1;
    if (e) x = df_mul(x, x);
  }
  return r;
}
__device__ __forceinline__ float df_round(df x) { return __fadd_rn(x.hi, x.lo); }
__device__ __forceinline__ df df_from_double(double x) {
  const float hi = float(x);
  return {hi, float(x - double(hi))};
}
__device__ __forceinline__ df df_shfl_down(df x, int d) {
  return {__shfl_down_sync(0xffffffffu, x.hi, d), __shfl_down_sync(0xffffffffu, x.lo, d)};
}
__device__ __forceinline__ df df_shfl(df x, int src) {
  return {__shfl_sync(0xffffffffu, x.hi, src), __shfl_sync(0xffffffffu, x.lo, src)};
}

// Coefficients of one recursion: a = gamma*lambda and g = gamma - a.
struct TC {
  df a, g;
};
// Per trajectory: the policy's (lambda_b) and, when the critic's recursion is
// not trivial, the critic's (lambda_critic). Table layout: [B][2] float4.
template <bool kCrit>
struct Coefs {
  TC p, c;
};
template <bool kCrit>
__device__ __forceinline__ Coefs<kCrit> load_coefs(const float4 *tab, int b) {
  Coefs<kCrit> k;
  const float4 u = __ldg(tab + 2 * b);
  k.p = {{u.x, u.y}, {u.z, u.w}};
  if constexpr (kCrit) {
    const float4 w = __ldg(tab + 2 * b + 1);
    k.c = {{w.x, w.y}, {w.z, w.w}};
  }
  return k;
}

// The affine map of a token segment, from the state at its right edge to the
// state at its left edge. fl bit 0: the segment holds the last token of a
// trajectory (the map ignores the incoming state); bit 1: the segment, left of
// any such end, holds an action token. Identity when fl == 0.
//   fl 1 (end, no action after it):  S' = (0, 0, 0, vp)          vp = reward waiting
//   fl 3 (end, then actions):         S' = (cp, cc, vp, 0)        vp = leftmost action value
//   fl 2 (actions, no end):           B' = ap (a B + g Vn + P) + cp,  Vn' = vp,  P' = 0
// with (a, g) = kp, the coefficients of the segment's trajectory.
template <bool kCrit>
struct CritMap {
  df ac, cc;
  TC kc;
};
template <>
struct CritMap<false> {};
template <bool kCrit>
struct GMap : CritMap<kCrit> {
  int fl;
  float vp;
  df ap, cp;
  TC kp;
};
struct GState {
  df Bp, Bc;
  float Vn, P;
};

template <bool kCrit>
__device__ __forceinline__ GMap<kCrit> identity_map() {
  GMap<kCrit> m;
  m.fl = 0;
  m.vp = 0.f;
  m.ap = m.cp = {0.f, 0.f};
  m.kp = {{0.f, 0.f}, {0.f, 0.f}};
  if constexpr (kCrit) {
    m.ac = m.cc = {0.f, 0.f};
    m.kc = {{0.f, 0.f}, {0.f, 0.f}};
  }
  return m;
}
__device__ __forceinline__ GState zero_state() {
  GState s;
  s.Bp = s.Bc = {0.f, 0.f};
  s.Vn = s.P = 0.f;
  return s;
}

// One action token's update of a lambda-return: a B + g Vn, or the waiting
// reward right after a trajectory end (where B = Vn = 0).
__device__ __forceinline__ df step_return(const TC &k, df B, float Vn, float P) {
  const df n = df_axpby(k.a, B, k.g, Vn);
  return P != 0.f ? df{P, 0.f} : n;
}

// x o y: x is the left segment, y the one immediately to its right.
template <bool kCrit>
__device__ GMap<kCrit> compose(const GMap<kCrit> &x, const GMap<kCrit> &y) {
  if (x.fl & 1) return x;
  if (!(x.fl & 2)) return y;
  if (!(y.fl & 3)) return x;
  const bool yact = (y.fl & 2) != 0;
  const float Yv = yact ? y.vp : 0.f, Yp = yact ? 0.f : y.vp;
  GMap<kCrit> r = x;
  r.cp = df_add(df_mul(x.ap, step_return(x.kp, y.cp, Yv, Yp)), x.cp);
  if constexpr (kCrit) r.cc = df_add(df_mul(x.ac, step_return(x.kc, y.cc, Yv, Yp)), x.cc);
  if (y.fl & 1) {
    r.fl = 3;
    r.ap = {0.f, 0.f};
    if constexpr (kCrit) r.ac = {0.f, 0.f};
  } else {  // same trajectory on both sides
    r.ap = df_mul(df_mul(x.ap, x.kp.a), y.ap);
    if constexpr (kCrit) r.ac = df_mul(df_mul(x.ac, x.kc.a), y.ac);
  }
  return r;
}

template <bool kCrit>
__device__ GState apply(const GMap<kCrit> &m, const GState &s) {
  GState r = zero_state();
  if (m.fl & 1) {
    const bool act = (m.fl & 2) != 0;
    r.Bp = m.cp;
    if constexpr (kCrit) r.Bc = m.cc;
    r.Vn = act ? m.vp : 0.f;
    r.P = act ? 0.f : m.vp;
    return r;
  }
  if (!(m.fl & 2)) return s;
  r.Bp = df_add(df_mul(m.ap, step_return(m.kp, s.Bp, s.Vn, s.P)), m.cp);
  if constexpr (kCrit) r.Bc = df_add(df_mul(m.ac, step_return(m.kc, s.Bc, s.Vn, s.P)), m.cc);
  r.Vn = m.vp;
  return r;
}

// The map of lane + d. compose reads the coefficients of its left operand
// only, so the scan's rounds leave them out (kCoefs = false: r's are the
// caller's own).
template <bool kCrit, bool kCoefs = true>
__device__ __forceinline__ GMap<kCrit> shfl_down_map(const GMap<kCrit> &m, int d) {
  GMap<kCrit> r = m;
  r.fl = __shfl_down_sync(0xffffffffu, m.fl, d);
  r.vp = __shfl_down_sync(0xffffffffu, m.vp, d);
  r.ap = df_shfl_down(m.ap, d);
  r.cp = df_shfl_down(m.cp, d);
  if constexpr (kCoefs) {
    r.kp.a = df_shfl_down(m.kp.a, d);
    r.kp.g = df_shfl_down(m.kp.g, d);
  }
  if constexpr (kCrit) {
    r.ac = df_shfl_down(m.ac, d);
    r.cc = df_shfl_down(m.cc, d);
    if constexpr (kCoefs) {
      r.kc.a = df_shfl_down(m.kc.a, d);
      r.kc.g = df_shfl_down(m.kc.g, d);
    }
  }
  return r;
}
__device__ __forceinline__ GState shfl_state(const GState &s, int src) {
  GState r;
  r.Bp = df_shfl(s.Bp, src);
  r.Bc = df_shfl(s.Bc, src);
  r.Vn = __shfl_sync(0xffffffffu, s.Vn, src);
  r.P = __shfl_sync(0xffffffffu, s.P, src);
  return r;
}

// ---------------------------------------------------------------------------
// cross-warp publication (decoupled look-back)
// ---------------------------------------------------------------------------
// Every published field is one naturally aligned 8-byte word: the field's 32
// bits and a tag (1) in the high half. An 8-byte access is single-copy atomic,
// so a reader that sees the tags of all words of a record has read the whole
// record, with no fence on either side and no separate status word: a poll is
// one round trip to L2. The arrays are zeroed before the scan, so an unwritten
// word reads as untagged.
constexpr uint64_t kTag = uint64_t(1) << 32;
template <bool kCrit>
constexpr int kMapWords = kCrit ? 18 : 10;  // GMap fields
template <bool kCrit>
constexpr int kStateWords = kCrit ? 6 : 4;  // GState fields

__device__ __forceinline__ void st_pair(uint64_t *p, float x, float y) {
  const uint64_t u = kTag | __float_as_uint(x), v = kTag | __float_as_uint(y);
  asm volatile("st.relaxed.gpu.global.v2.b64 [%0], {%1, %2};" ::"l"(p), "l"(u), "l"(v) : "memory");
}
// True when both words carry the tag.
__device__ __forceinline__ bool ld_pair(const uint64_t *p, float &x, float &y) {
  uint64_t u, v;
  asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(u), "=l"(v) : "l"(p) : "memory");
  x = __uint_as_float(uint32_t(u));
  y = __uint_as_float(uint32_t(v));
  return ((u & v) >> 32) != 0;
}
__device__ __forceinline__ bool ld_pair(const uint64_t *p, df &x) { return ld_pair(p, x.hi, x.lo); }

template <bool kCrit>
__device__ void publish_map(uint64_t *p, const GMap<kCrit> &m) {
  st_pair(p + 0, __int_as_float(m.fl), m.vp);
  st_pair(p + 2, m.ap.hi, m.ap.lo);
  st_pair(p + 4, m.cp.hi, m.cp.lo);
  st_pair(p + 6, m.kp.a.hi, m.kp.a.lo);
  st_pair(p + 8, m.kp.g.hi, m.kp.g.lo);
  if constexpr (kCrit) {
    st_pair(p + 10, m.ac.hi, m.ac.lo);
    st_pair(p + 12, m.cc.hi, m.cc.lo);
    st_pair(p + 14, m.kc.a.hi, m.kc.a.lo);
    st_pair(p + 16, m.kc.g.hi, m.kc.g.lo);
  }
}
template <bool kCrit>
__device__ bool fetch_map(const uint64_t *p, GMap<kCrit> &m) {
  float f;
  bool ok = ld_pair(p + 0, f, m.vp);
  m.fl = __float_as_int(f);
  ok &= ld_pair(p + 2, m.ap);
  ok &= ld_pair(p + 4, m.cp);
  ok &= ld_pair(p + 6, m.kp.a);
  ok &= ld_pair(p + 8, m.kp.g);
  if constexpr (kCrit) {
    ok &= ld_pair(p + 10, m.ac);
    ok &= ld_pair(p + 12, m.cc);
    ok &= ld_pair(p + 14, m.kc.a);
    ok &= ld_pair(p + 16, m.kc.g);
  }
  return ok;
}
template <bool kCrit>
__device__ void publish_state(uint64_t *p, const GState &s) {
  st_pair(p + 0, s.Bp.hi, s.Bp.lo);
  st_pair(p + 2, s.Vn, s.P);
  if constexpr (kCrit) st_pair(p + 4, s.Bc.hi, s.Bc.lo);
}
template <bool kCrit>
__device__ bool fetch_state(const uint64_t *p, GState &s) {
  bool ok = ld_pair(p + 0, s.Bp);
  ok &= ld_pair(p + 2, s.Vn, s.P);
  if constexpr (kCrit) ok &= ld_pair(p + 4, s.Bc);
  else s.Bc = {0.f, 0.f};
  return ok;
}

struct GaeArgs {
  const float *values, *rewards;
  const uint8_t *m;
  const int32_t *cu;
  int B;
  int64_t N;
  int nchunks;             // scan chunks of 32 lanes x seg tokens
  int pieces;              // 32-token pieces per lane segment (1, 2 or 4)
  int nsub;                // 1024-token sub-chunks, the units of chunk_first
  const float4 *coef;      // [B][2]
  const int *chunk_first;  // [nsub] trajectory of each 1024-token sub-chunk's first token
  int *ticket;
  uint64_t *agg;           // [nchunks][kMapWords]: map of the whole chunk
  uint64_t *incl;          // [nchunks][kStateWords]: state at the chunk's left edge
  float *adv, *ret;
  unsigned int *err;
  uint64_t wait_ns;        // bound of every look-back wait
  int64_t tma_rows;        // lane-segment rows the tensor maps cover (0: no maps)
};

// The per-token arrays viewed as [tma_rows][seg] (a row per lane segment),
// box 32 x 32 (one piece of one chunk), swizzled as the staging layout below:
// values, advantages and returns in 128-byte rows by row mod 8, the mask in
// 32-byte rows by bit 2 of the row.
struct ScanMaps {
  CUtensorMap v, m, adv, ret;
};

using seg::CuView;



// State at the right edge of chunk q, from the chunks to its right. The warp
// polls the 32 successors q+1 .. q+32, each lane one chunk's published state
// and map, until the first chunk whose left-edge state is known (published
// state, a map that ignores its right neighbour, or the end of the input) lies
// in that window with every map before it published; the state then goes
// through the maps of the chunks before it one by one. Every state is thus
// the same chain of map applications from the nearest trajectory end, however
// the warps were timed, and the results are bit-identical from run to run.
// The wait ends: the highest unfinished chunk only waits on finished ones.
// Every wait is bounded.
template <bool kCrit>
__device__ GState look_back(const GaeArgs &a, int q, int lane) {
  const uint64_t t_start = globaltimer_ns();
  const int j = q + 1 + lane;
  GMap<kCrit> mj = identity_map<kCrit>();
  GState sj = zero_state();
  int kind = 2;  // 0: nothing published yet, 1: map, 2: left-edge state known
  uint32_t polls = 0;
  int stop;
  for (;;) {
    if (j < a.nchunks) {
      const bool has_s = fetch_state<kCrit>(a.incl + size_t(j) * kStateWords<kCrit>, sj);
      const bool has_m = fetch_map<kCrit>(a.agg + size_t(j) * kMapWords<kCrit>, mj);
      kind = has_s ? 2 : (has_m ? 1 : 0);
      if (kind == 1 && (mj.fl & 1)) {  // the map ignores its right neighbour
        sj = apply<kCrit>(mj, zero_state());
        kind = 2;
      }
    }
    const unsigned bt = __ballot_sync(0xffffffffu, kind == 2);
    const unsigned bn = __ballot_sync(0xffffffffu, kind == 0);
    stop = bt ? __ffs(bt) - 1 : 32;
    const int first_nr = bn ? __ffs(bn) - 1 : 32;
    if (stop < 32 && first_nr > stop) break;  // a known state, and every map before it
    if ((++polls & 31u) == 0u && globaltimer_ns() - t_start > a.wait_ns) {
      if (lane == 0) raise_device_error(a.err, SAO_DEVERR_SCAN_TIMEOUT);
      return zero_state();
    }
    __nanosleep(64);
  }
  // carry the known state through the maps of lanes stop-1 .. 0
  GState cur = shfl_state(sj, stop);
  for (int i = stop - 1; i >= 0; --i) cur = shfl_state(apply<kCrit>(mj, cur), i);
  return cur;
}

// ---------------------------------------------------------------------------
// per-warp staging in shared memory
// ---------------------------------------------------------------------------
// A scan chunk is 32 lane segments of seg = 32 * pieces consecutive tokens;
// lane r's segment starts at chunk offset r * seg. The fold streams the
// segments through shared memory one 32-token piece at a time (right to
// left): row r of a staged piece holds lane r's 32 tokens of that piece.
// val rows are 8 granules of 16 bytes, granule j stored at
// 8r + (j ^ (r & 7)) (the tensor copies' 128-byte swizzle, buffers 1024-byte
// aligned); msk rows are 2 granules, granule j at 2r + (j ^ ((r >> 2) & 1))
// (their 32-byte swizzle). 8 lanes reading the same granule of their own
// rows then touch 8 distinct bank groups. The two value buffers hold the
// piece being folded and the next one, copied meanwhile; chunks the tensor
// maps do not cover (the ragged end, unaligned arrays) are staged element by
// element in the same layout. Each lane also stores its values into its own TMEM
// lane (the warp's 32 lanes of the CTA's allocation, column 32 (s + k) + i for
// token i of piece k, where the slot s is 0, or 2 for the second of two
// 2-piece chunks in flight) and its action bits into act[s + k] (the chunk's
// trajectory-end bits are in ends[s + k]), so that the replay, after the
// look-back, reads the chunk from the SM instead of from DRAM a second time;
// the replay writes advantages into val[0] and returns into val[1], which two
// tensor stores take out.
constexpr int kScanCuCap = 120;   // cu_seqlens entries staged per warp
constexpr int kScanTrajCap = 32;  // trajectories whose coefficients and reward are staged per warp
struct __align__(16) WarpBuf {
  float val[2][kChunk];           // values of two pieces (fold); advantages and returns of one (replay)
  uint8_t msk[kChunk];            // action flags of the piece being copied
  uint32_t act[kMaxPieces][32];   // per piece, each lane's action bits
  uint32_t ends[kMaxPieces][32];  // per piece, each lane's trajectory-end bits
  int32_t cu[kScanCuCap];         // cu_seqlens slice of the chunk being folded
  float4 coef[kScanTrajCap][2];   // its trajectories' coefficient rows
  float rew[kScanTrajCap];        // and rewards
  uint64_t bar[2];                // completion of the tensor copies into val[0] / val[1]
  int abort;                      // a copy did not complete in time
  uint32_t tmem;                  // TMEM address of the CTA's allocation (warp 0's buffer)
};
// Each warp's buffer starts 1024-byte aligned (the 128-byte swizzle's period)
constexpr size_t kWarpBufBytes = (sizeof(WarpBuf) + 1023) / 1024 * 1024;
__device__ __forceinline__ TC coef_row(float4 u) { return {{u.x, u.y}, {u.z, u.w}}; }

// Coefficients and reward of trajectory b: from the warp's staged copy when
// the chunk's trajectories fit, else from global memory.
struct TrajView {
  const float4 *gcoef;
  const float *grew;
  const float4 (*scoef)[2];
  const float *srew;
  int blo;
  bool in_smem;
  template <bool kCrit>
  __device__ __forceinline__ Coefs<kCrit> coefs(int b) const {
    if (!in_smem) return load_coefs<kCrit>(gcoef, b);
    Coefs<kCrit> k;
    k.p = coef_row(scoef[b - blo][0]);
    if constexpr (kCrit) k.c = coef_row(scoef[b - blo][1]);
    return k;
  }
  __device__ __forceinline__ float reward(int b) const { return in_smem ? srew[b - blo] : __ldg(grew + b); }
};
__device__ __forceinline__ int fgran(int r, int j) { return 8 * r + (j ^ (r & 7)); }
__device__ __forceinline__ int mgran(int r, int j) { return 2 * r + (j ^ ((r >> 2) & 1)); }

// The lane's 4 TMEM columns from `taddr` (lane field: the warp's TMEM lanes).
__device__ __forceinline__ void tmem_st4(uint32_t taddr, float4 v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr),
               "r"(__float_as_uint(v.x)), "r"(__float_as_uint(v.y)), "r"(__float_as_uint(v.z)),
               "r"(__float_as_uint(v.w))
               : "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// Starts the load of 4 TMEM columns; the registers hold them only after
// tmem_wait_ld4 on the same registers (which the compiler then cannot read
// earlier).
__device__ __forceinline__ void tmem_ld4(uint32_t taddr, uint32_t (&r)[4]) {
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(taddr)
               : "memory");
}
__device__ __forceinline__ void tmem_wait_ld4(uint32_t (&r)[4]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3])::"memory");
}

// The tensor copies of a piece, with an L2 policy (every input line is read
// once: the copies leave L2 first).
__device__ __forceinline__ void tma_load_hint(uint32_t dst, const CUtensorMap *map, uint32_t bar, int32_t x, int32_t y,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%3, "
      "%4}], [%2], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y), "l"(policy)
      : "memory");
}

// Whether chunk q lies in the rows the tensor maps cover.
__device__ __forceinline__ bool chunk_tma(const GaeArgs &a, int q) { return 32 * (int64_t(q) + 1) <= a.tma_rows; }

// Starts the copy of piece k of chunk q (first token c0) into val and msk:
// one tensor copy each when the chunk has them (completion on `bar`),
// element by element otherwise (zero past N).
__device__ __forceinline__ void stage_in(const GaeArgs &a, const ScanMaps &mp, bool tma, int q, int64_t c0, int seg,
                                         int k, int lane, float *val, uint8_t *msk, uint32_t bar, uint64_t policy) {
  if (tma) {
    if (lane == 0) {
      tc::mbar_arrive_expect_tx(bar, uint32_t(kChunk * (sizeof(float) + 1)));
      tma_load_hint(tc::smem_u32(val), &mp.v, bar, 32 * k, 32 * q, policy);
      tma_load_hint(tc::smem_u32(msk), &mp.m, bar, 32 * k, 32 * q, policy);
    }
    return;
  }
  const int64_t N = a.N;
  const int64_t off = c0 + 32 * int64_t(k);
#pragma unroll 1
  for (int i = lane; i < kChunk; i += 32) {
    const int r = i >> 5, kk = i & 31;
    const int64_t t = off + int64_t(r) * seg + kk;
    val[4 * fgran(r, kk >> 2) + (kk & 3)] = t < N ? a.values[t] : 0.f;
    msk[16 * mgran(r, kk >> 4) + (kk & 15)] = (t < N && a.m[t] != 0) ? 1 : 0;
  }
}

// Waits for the piece staged into buffer `buf` (parity bit buf of `phases`).
__device__ __forceinline__ void stage_wait(const GaeArgs &a, bool tma, WarpBuf &w, int buf, uint32_t &phases) {
  if (tma) {
    tc::mbar_wait(tc::smem_u32(&w.bar[buf]), (phases >> buf) & 1u, &w.abort, a.err);
    phases ^= 1u << buf;
  }
  __syncwarp();
}

// Stores piece k of chunk q from val (advantages) and ret (returns); on
// return the buffers may be written again.
__device__ __forceinline__ void stage_out(const GaeArgs &a, const ScanMaps &mp, bool tma, int q, int64_t c0, int seg,
                                          int k, int lane, const float *val, const float *ret, uint64_t policy) {
  if (tma) {
    tc::fence_proxy_async_smem();  // this lane's writes, visible to the tensor copy
    __syncwarp();
    if (lane == 0) {
      tc::tma_store_2d_hint(&mp.adv, tc::smem_u32(val), 32 * k, 32 * q, policy);
      tc::tma_store_2d_hint(&mp.ret, tc::smem_u32(ret), 32 * k, 32 * q, policy);
      tc::bulk_commit_group();
      tc::bulk_wait_group_read<0>();
    }
    __syncwarp();
    return;
  }
  const int64_t N = a.N;
  const int64_t off = c0 + 32 * int64_t(k);
#pragma unroll 1
  for (int i = lane; i < kChunk; i += 32) {
    const int r = i >> 5, kk = i & 31;
    const int64_t t = off + int64_t(r) * seg + kk;
    if (t < N) {
      a.adv[t] = val[4 * fgran(r, kk >> 2) + (kk & 3)];
      a.ret[t] = ret[4 * fgran(r, kk >> 2) + (kk & 3)];
    }
  }
  tc::fence_proxy_async_smem();  // these reads before a later tensor copy into the buffers
  __syncwarp();
}

// Bit i set when byte i of x is non-zero (i = 0..3).
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t x) {
  const uint32_t h = (((x & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | x) & 0x80808080u;
  return (h * 0x00204081u) >> 28;
}

// Action-token bits of the lane's staged row (bit k: token k of the piece).
__device__ __forceinline__ uint32_t row_actions(const uint8_t *msk, int lane) {
  const uint4 m0 = *reinterpret_cast<const uint4 *>(&msk[16 * mgran(lane, 0)]);
  const uint4 m1 = *reinterpret_cast<const uint4 *>(&msk[16 * mgran(lane, 1)]);
  return nonzero_bytes(m0.x) | nonzero_bytes(m0.y) << 4 | nonzero_bytes(m0.z) << 8 | nonzero_bytes(m0.w) << 12 |
         nonzero_bytes(m1.x) << 16 | nonzero_bytes(m1.y) << 20 | nonzero_bytes(m1.z) << 24 |
         nonzero_bytes(m1.w) << 28;
}

// The trajectory ends of the chunk at c0 (pieces pieces in `slot`), as bits:
// every end e = cu[b + 1] - 1 inside the chunk sets bit u mod 32 of
// ends[slot + u / 32][r], where r = (e - c0) / seg and u = (e - c0) mod seg.
__device__ __forceinline__ void mark_ends(const CuView &cu, int blo, int bhi, int64_t c0, int seg, int pieces,
                                          int slot, int lane, WarpBuf &w) {
#pragma unroll 1
  for (int i = lane; i < 32 * pieces; i += 32) w.ends[slot + (i >> 5)][i & 31] = 0u;
  __syncwarp();
  const int64_t c1 = c0 + 32 * int64_t(seg);
  const int lseg = 31 - __clz(seg);  // seg is a power of two
#pragma unroll 1
  for (int b = blo + lane; b <= bhi; b += 32) {
    const int64_t e = cu[b + 1] - 1;
    if (e >= c0 && e < c1) {
      const int off = int(e - c0), u = off & (seg - 1);
      atomicOr(&w.ends[slot + (u >> 5)][off >> lseg], 1u << (u & 31));
    }
  }
  __syncwarp();
}

// ---------------------------------------------------------------------------
// per-lane fold and replay
// ---------------------------------------------------------------------------
// A piece's tokens are t0 .. t0+31; bit k of `act` / `ends`: token t0+k is an
// action token / the last token of its trajectory; blo .. bhi bound the
// trajectories the chunk can touch.

// The token loops below take 4 tokens at a time. A group in which no lane of
// the warp holds a trajectory end (the common case: trajectories span
// thousands of tokens) runs branch-free, one fused double-float a*B + g*V per
// token with the action flag applied by selects; otherwise the warp takes the
// general path for that group. A reward still waiting for its action token
// (observation tokens after a trajectory's last action token) rides along on
// the branch-free path: there B = Vn = 0, the step's products and sums are
// exactly 0, and adding the reward to the high part gives the (R, 0) of the
// general path's step.

// A lane's fold of its segment so far (the pieces right of the current one):
// the lambda-returns with a zero state at the segment's right edge, the value
// of the leftmost action token folded, the reward still waiting, the map
// flags and the number of action tokens.
template <bool kCrit>
struct FoldState {
  Coefs<kCrit> k;
  df Bp, Bc;
  float Vn, P;
  int fl, nact;
};

template <bool kCrit>
__device__ void fold_piece(const GaeArgs &a, const float *val, uint32_t tcol, int lane, uint32_t act, uint32_t ends,
                           int64_t t0, const CuView &cu, const TrajView &tv, int blo, int bhi,
                           FoldState<kCrit> &f) {
  Coefs<kCrit> k = f.k;
  df Bp = f.Bp, Bc = f.Bc;
  float Vn = f.Vn, P = f.P;
  int fl = f.fl;
  const int sw = lane & 7;
  const bool any_end = __any_sync(0xffffffffu, ends != 0u);  // else no group needs the general path
#pragma unroll 1
  for (int g = 7; g >= 0; --g) {
    const float4 v4 = *reinterpret_cast<const float4 *>(&val[4 * (8 * lane + (g ^ sw))]);
    tmem_st4(tcol + 4 * g, v4);  // kept for the replay
    const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
    const uint32_t a4 = (act >> (4 * g)) & 15u, e4 = (ends >> (4 * g)) & 15u;
    if (any_end && __any_sync(0xffffffffu, e4 != 0u)) {
#pragma unroll 1
      for (int i = 3; i >= 0; --i) {
        const float v = i == 3 ? vv[3] : (i == 2 ? vv[2] : (i == 1 ? vv[1] : vv[0]));
        if ((e4 >> i) & 1u) {  // last token of a trajectory: reset
          const int b = cu.find(blo, bhi, t0 + 4 * g + i);
          k = tv.coefs<kCrit>(b);
          P = tv.reward(b);
          Bp = Bc = {0.f, 0.f};
          Vn = 0.f;
          fl = 1;
        }
        if ((a4 >> i) & 1u) {
          Bp = step_return(k.p, Bp, Vn, P);
          if constexpr (kCrit) Bc = step_return(k.c, Bc, Vn, P);
          Vn = v;
          P = 0.f;
          fl |= 2;
        }
      }
    } else {
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        const bool on = (a4 >> i) & 1u;
        df np = df_axpby_u(k.p.a, Bp, k.p.g, Vn);
        np.hi = __fadd_rn(np.hi, P);
        Bp = on ? np : Bp;
        if constexpr (kCrit) {
          df nc = df_axpby_u(k.c.a, Bc, k.c.g, Vn);
          nc.hi = __fadd_rn(nc.hi, P);
          Bc = on ? nc : Bc;
        }
        Vn = on ? vv[i] : Vn;
        P = on ? 0.f : P;
      }
      fl |= a4 ? 2 : 0;
    }
  }
  f.k = k;
  f.Bp = df_renorm(Bp);
  if constexpr (kCrit) Bc = df_renorm(Bc);
  f.Bc = Bc;
  f.Vn = Vn;
  f.P = P;
  f.fl = fl;
  f.nact += __popc(act);
}

// The map of the lane's whole segment from its fold.
template <bool kCrit>
__device__ GMap<kCrit> lane_map(const FoldState<kCrit> &f) {
  GMap<kCrit> m;
  m.fl = f.fl;
  m.vp = (f.fl & 2) ? f.Vn : f.P;
  m.cp = f.Bp;
  m.kp = f.k.p;
  // with no trajectory end every action token of the segment is in one trajectory
  m.ap = f.fl == 2 ? df_pow(f.k.p.a, f.nact - 1) : df{0.f, 0.f};
  if constexpr (kCrit) {
    m.cc = f.Bc;
    m.kc = f.k.c;
    m.ac = f.fl == 2 ? df_pow(f.k.c.a, f.nact - 1) : df{0.f, 0.f};
  }
  return m;
}

// A - V rounded to float, from the double-float lambda-return B: B.hi - V is
// exact when the two are within a factor of two of each other (the case where
// A is small against V), and otherwise already within half an ulp of A.
__device__ __forceinline__ float adv_round(df B, float v) { return __fadd_rn(__fsub_rn(B.hi, v), B.lo); }

// A lane's replay state: the state at the right edge of the current piece and
// the coefficients and reward of the trajectory there.
template <bool kCrit>
struct ReplayState {
  GState st;
  Coefs<kCrit> k;
  float R;
};

// Replays one piece from the values the fold left in TMEM (the next group's
// load in flight while a group is replayed); advantages go to the lane's row
// of `adv`, returns to its row of `ret`.
template <bool kCrit>
__device__ void replay_piece(const GaeArgs &a, uint32_t tcol, float *adv, float *ret, int lane, uint32_t act,
                             uint32_t ends, int64_t t0, const CuView &cu, const TrajView &tv, int blo, int bhi,
                             ReplayState<kCrit> &rs) {
  Coefs<kCrit> k = rs.k;
  float R = rs.R;
  GState st = rs.st;
  const int sw = lane & 7;
  const bool any_end = __any_sync(0xffffffffu, ends != 0u);  // else no group needs the general path
  uint32_t nx[4];
  tmem_ld4(tcol + 28, nx);
  tmem_wait_ld4(nx);
#pragma unroll 1
  for (int g = 7; g >= 0; --g) {
    float4 *vp = reinterpret_cast<float4 *>(&adv[4 * (8 * lane + (g ^ sw))]);
    float4 *rp = reinterpret_cast<float4 *>(&ret[4 * (8 * lane + (g ^ sw))]);
    const float vv[4] = {__uint_as_float(nx[0]), __uint_as_float(nx[1]), __uint_as_float(nx[2]),
                         __uint_as_float(nx[3])};
    if (g > 0) tmem_ld4(tcol + 4 * (g - 1), nx);
    float ov[4], orr[4];
    const uint32_t a4 = (act >> (4 * g)) & 15u, e4 = (ends >> (4 * g)) & 15u;
    if (any_end && __any_sync(0xffffffffu, e4 != 0u)) {
#pragma unroll 1
      for (int i = 3; i >= 0; --i) {
        const float v = i == 3 ? vv[3] : (i == 2 ? vv[2] : (i == 1 ? vv[1] : vv[0]));
        float o = 0.f, orv = 0.f;
        if ((e4 >> i) & 1u) {
          const int b = cu.find(blo, bhi, t0 + 4 * g + i);
          k = tv.coefs<kCrit>(b);
          R = tv.reward(b);
          st.Bp = st.Bc = {0.f, 0.f};
          st.Vn = 0.f;
          st.P = R;
        }
        if ((a4 >> i) & 1u) {
          st.Bp = step_return(k.p, st.Bp, st.Vn, st.P);
          if constexpr (kCrit) st.Bc = step_return(k.c, st.Bc, st.Vn, st.P);
          o = adv_round(st.Bp, v);
          // gamma = lambda_critic = 1: the critic's return is the trajectory's reward
          orv = kCrit ? df_round(st.Bc) : R;
          st.Vn = v;
          st.P = 0.f;
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          ov[j] = j == i ? o : ov[j];
          orr[j] = j == i ? orv : orr[j];
        }
      }
    } else {
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        const bool on = (a4 >> i) & 1u;
        df np = df_axpby_u(k.p.a, st.Bp, k.p.g, st.Vn);
        np.hi = __fadd_rn(np.hi, st.P);
        ov[i] = on ? adv_round(np, vv[i]) : 0.f;
        st.Bp = on ? np : st.Bp;
        if constexpr (kCrit) {
          df nc = df_axpby_u(k.c.a, st.Bc, k.c.g, st.Vn);
          nc.hi = __fadd_rn(nc.hi, st.P);
          orr[i] = on ? df_round(nc) : 0.f;
          st.Bc = on ? nc : st.Bc;
        } else {
          orr[i] = on ? R : 0.f;
        }
        st.Vn = on ? vv[i] : st.Vn;
        st.P = on ? 0.f : st.P;
      }
    }
    *vp = make_float4(ov[0], ov[1], ov[2], ov[3]);
    *rp = make_float4(orr[0], orr[1], orr[2], orr[3]);
    if (g > 0) tmem_wait_ld4(nx);
  }
  rs.k = k;
  rs.R = R;
  st.Bp = df_renorm(st.Bp);
  if constexpr (kCrit) st.Bc = df_renorm(st.Bc);
  rs.st = st;
}

// What a lane keeps about a folded chunk for its look-back and replay.
template <bool kCrit>
struct Pending {
  int q;           // chunk index
  int slot;        // TMEM columns from 32 * slot and act rows from slot hold the chunk
  int blo, bhi;    // trajectories the chunk can touch
  int b_seg;       // trajectory of the lane's last token below N
  GMap<kCrit> E;   // maps of the lanes to the right within the chunk
  GMap<kCrit> S;   // lane 0: map of the whole chunk
};

__device__ __forceinline__ int take_chunk(const GaeArgs &a, int lane) {
  int t = 0;
  if (lane == 0) t = atomicAdd(a.ticket, 1);
  return a.nchunks - 1 - __shfl_sync(0xffffffffu, t, 0);
}

// Folds each lane's segment of chunk q piece by piece (right to left, the
// next piece copied while the current one is folded and its values kept in
// TMEM), scans the lane maps and publishes the chunk's map (or, when it
// ignores its right neighbour, its left-edge state). Nothing here waits on
// another warp.
template <bool kCrit>
__device__ void fold_chunk(const GaeArgs &a, const ScanMaps &mp, WarpBuf &w, uint32_t tmem, int lane, int q, int slot,
                           uint32_t &phases, Pending<kCrit> &p) {
  const int seg = 32 * a.pieces;
  const int64_t c0 = int64_t(q) * kChunk * a.pieces;
  const int64_t s0 = c0 + int64_t(lane) * seg;  // the lane's segment
  const int64_t N = a.N;
  const bool tma = chunk_tma(a, q);
  const uint64_t pol = tc::l2_evict_first();
  tc::fence_proxy_async_smem();  // this lane's reads of val and msk before the copies refill them
  __syncwarp();
  stage_in(a, mp, tma, q, c0, seg, a.pieces - 1, lane, w.val[0], w.msk, tc::smem_u32(&w.bar[0]), pol);

  // This chunk's slice of cu_seqlens, in shared memory when it fits.
  const int sub0 = q * a.pieces, sub1 = (q + 1) * a.pieces;
  const int blo = __ldg(a.chunk_first + sub0);
  const int bhi = sub1 < a.nsub ? __ldg(a.chunk_first + sub1) : a.B - 1;
  const int ncu = bhi - blo + 2;  // cu[blo .. bhi + 1]
  const CuView cu{a.cu, w.cu, blo, ncu <= kScanCuCap};
  const TrajView tv{a.coef, a.rewards, w.coef, w.rew, blo, ncu - 1 <= kScanTrajCap};
  if (cu.in_smem)
    for (int i = lane; i < ncu; i += 32) w.cu[i] = __ldg(a.cu + blo + i);
  if (tv.in_smem && lane < ncu - 1) {  // with the cu_seqlens slice, in one round trip
    w.coef[lane][0] = __ldg(a.coef + 2 * (blo + lane));
    if constexpr (kCrit) w.coef[lane][1] = __ldg(a.coef + 2 * (blo + lane) + 1);
    w.rew[lane] = __ldg(a.rewards + blo + lane);
  }
  __syncwarp();
  mark_ends(cu, blo, bhi, c0, seg, a.pieces, slot, lane, w);

  // the trajectory of the lane's last token below N gives its first coefficients
  const int64_t s_end = (s0 + seg < N ? s0 + seg : N) - 1;
  const int b_seg = s0 < N ? cu.find(blo, bhi, s_end) : blo;
  FoldState<kCrit> f;
  f.k = tv.coefs<kCrit>(b_seg);
  f.Bp = f.Bc = {0.f, 0.f};
  f.Vn = f.P = 0.f;
  f.fl = 0;
  f.nact = 0;
#pragma unroll 1
  for (int k = a.pieces - 1; k >= 0; --k) {
    const int cur = (a.pieces - 1 - k) & 1;
    stage_wait(a, tma, w, cur, phases);
    const uint32_t act = row_actions(w.msk, lane);
    w.act[slot + k][lane] = act;
    tc::fence_proxy_async_smem();  // the reads of msk and of the other value buffer before the next copy
    __syncwarp();  // every lane has read the flags and finished the previous piece
    if (k > 0)
      stage_in(a, mp, tma, q, c0, seg, k - 1, lane, w.val[cur ^ 1], w.msk, tc::smem_u32(&w.bar[cur ^ 1]), pol);
    const int64_t t0 = s0 + 32 * int64_t(k);
    // every lane folds (the token loops vote across the warp); a lane past N
    // has no flags and keeps its state
    fold_piece<kCrit>(a, w.val[cur], tmem + 32 * (slot + k), lane, act, w.ends[slot + k][lane], t0, cu, tv, blo, bhi,
                      f);
  }
  tmem_wait_st();  // the values are in TMEM before the replay reads them

  // the suffix scan of the warp's 32 lane maps
  GMap<kCrit> S = lane_map<kCrit>(f);
#pragma unroll 1
  for (int d = 1; d < 32; d <<= 1) {
    const GMap<kCrit> o = shfl_down_map<kCrit, false>(S, d);
    if (lane + d < 32) S = compose<kCrit>(S, o);
  }
  GMap<kCrit> E = shfl_down_map<kCrit>(S, 1);  // lanes to my right within the chunk
  if (lane == 31) E = identity_map<kCrit>();

  // A chunk whose map ignores its right neighbour publishes its left-edge
  // state at once; the others publish their map.
  if (lane == 0) {
    if (q == a.nchunks - 1 || (S.fl & 1))
      publish_state<kCrit>(a.incl + size_t(q) * kStateWords<kCrit>, apply<kCrit>(S, zero_state()));
    else
      publish_map<kCrit>(a.agg + size_t(q) * kMapWords<kCrit>, S);
  }
  p.q = q;
  p.slot = slot;
  p.blo = blo;
  p.bhi = bhi;
  p.b_seg = b_seg;
  p.E = E;
  p.S = S;
}

// Looks back for the state at the chunk's right edge, publishes its left-edge
// state, then replays the tokens piece by piece (right to left) from TMEM and
// stores advantages and returns.
template <bool kCrit>
__device__ int replay_chunk(const GaeArgs &a, const ScanMaps &mp, WarpBuf &w, uint32_t tmem, int lane,
                            const Pending<kCrit> &p, bool pipelined) {
  const int seg = 32 * a.pieces;
  const int64_t c0 = int64_t(p.q) * kChunk * a.pieces;
  const int64_t s0 = c0 + int64_t(lane) * seg;
  const bool last = (p.q == a.nchunks - 1);
  const bool reset = __shfl_sync(0xffffffffu, p.S.fl & 1, 0) != 0;  // lane 0 holds the chunk's map
  // Unless the next chunk has been folded since, the fold's copies of the
  // chunk's cu_seqlens slice and trajectory table are still in shared memory.
  const CuView cu{a.cu, w.cu, p.blo, !pipelined && p.bhi - p.blo + 2 <= kScanCuCap};
  const TrajView tv{a.coef, a.rewards, w.coef, w.rew, p.blo, !pipelined && p.bhi - p.blo + 1 <= kScanTrajCap};
  // the coefficients and reward of the lane's last trajectory, loaded while
  // the look-back runs
  ReplayState<kCrit> rs;
  rs.k = tv.coefs<kCrit>(p.b_seg);
  rs.R = tv.reward(p.b_seg);
  GState right = zero_state();
  if (!last) right = look_back<kCrit>(a, p.q, lane);
  if (lane == 0 && !reset && !last)
    publish_state<kCrit>(a.incl + size_t(p.q) * kStateWords<kCrit>, apply<kCrit>(p.S, right));
  // every lane replays (the token loops vote across the warp); rows past N
  // are never stored
  rs.st = apply<kCrit>(p.E, right);
  const bool tma = chunk_tma(a, p.q);
  const uint64_t pol = tc::l2_evict_first();
  int t = 0;
#pragma unroll 1
  for (int k = a.pieces - 1; k >= 0; --k) {
    // one chunk at a time: the next ticket is taken before the last piece so
    // that its round trip overlaps the piece. The chunk is folded right after
    // this replay, which waits on nothing, so the tickets still only wait on
    // chunks that are folded without waiting.
    if (!pipelined && k == 0 && lane == 0) t = atomicAdd(a.ticket, 1);
    const uint32_t act = w.act[p.slot + k][lane];
    const int64_t t0 = s0 + 32 * int64_t(k);
    replay_piece<kCrit>(a, tmem + 32 * (p.slot + k), w.val[0], w.val[1], lane, act, w.ends[p.slot + k][lane], t0,
                        cu, tv, p.blo, p.bhi, rs);
    __syncwarp();
    stage_out(a, mp, tma, p.q, c0, seg, k, lane, w.val[0], w.val[1], pol);
  }
  return pipelined ? -1 : a.nchunks - 1 - __shfl_sync(0xffffffffu, t, 0);
}

// Persistent warps: a warp takes a chunk (ticket), folds and publishes it,
// looks back and replays it. Tickets keep the decoupled look-back safe: a
// warp waits only on chunks taken before its own, and every taken chunk is
// folded and published at once, before its warp waits on anything. Each CTA
// holds kTmemCols TMEM columns for the whole launch (four CTAs per SM take all
// 512, so the allocation never waits on this kernel).
template <bool kCrit, bool kPipe>
__global__ void __launch_bounds__(kThreads, kMinBlocks)
    gae_scan_kernel(GaeArgs a, const __grid_constant__ ScanMaps mp) {
  extern __shared__ __align__(1024) unsigned char s_raw[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t raw = tc::smem_u32(s_raw);
  unsigned char *base = s_raw + (((raw + 1023u) & ~1023u) - raw);
  WarpBuf &w = *reinterpret_cast<WarpBuf *>(base + size_t(warp) * kWarpBufBytes);
  WarpBuf &w0 = *reinterpret_cast<WarpBuf *>(base);
  if (lane == 0) {
    tc::mbar_init(tc::smem_u32(&w.bar[0]), 1);
    tc::mbar_init(tc::smem_u32(&w.bar[1]), 1);
    w.abort = 0;
    tc::fence_barrier_init();
  }
  uint32_t phases = 0;
  if (warp == 0) {
    tc::tmem_alloc(tc::smem_u32(&w0.tmem), kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = w0.tmem + (uint32_t(32 * warp) << 16);  // the warp's TMEM lanes
  if constexpr (kPipe) {
    // short segments: two chunks in flight, one per half of the warp's TMEM
    // columns; the warp folds a chunk before it looks back for the one it
    // folded before, so the chunks it waits on have had a whole fold to
    // publish (with one chunk at a time that wait is exposed, and at these
    // chunk sizes it dominates)
    // (one call site each for the fold and the replay: the kernel's code
    // stays small enough for the instruction cache)
    Pending<kCrit> p;
    bool have = false;
    int half = 0;
#pragma unroll 1
    for (int q = take_chunk(a, lane);; q = take_chunk(a, lane)) {
      Pending<kCrit> n;
      if (q >= 0) fold_chunk<kCrit>(a, mp, w, tmem, lane, q, half * (kMaxPieces / 2), phases, n);
      if (have) replay_chunk<kCrit>(a, mp, w, tmem, lane, p, true);
      if (q < 0) break;
      p = n;
      have = true;
      half ^= 1;
    }
  } else {
    // long segments: one chunk at a time in all of the warp's columns (the
    // per-chunk scan, look-back and set-up spread over 4096 tokens cost less
    // than the exposed wait)
#pragma unroll 1
    for (int q = take_chunk(a, lane); q >= 0;) {
      Pending<kCrit> p;
      fold_chunk<kCrit>(a, mp, w, tmem, lane, q, 0, phases, p);
      q = replay_chunk<kCrit>(a, mp, w, tmem, lane, p, false);  // takes the next ticket
    }
  }
  if (lane == 0) tc::bulk_wait_group<0>();  // the last stores are done
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(w0.tmem, kTmemCols);
  }
}

// Test hook: the scan's first `skip` tickets are taken before any warp runs,
// so the top chunks are never processed and the chunks below them wait for
// states that never come (until the bounded wait gives up).
__global__ void preset_ticket_kernel(int *ticket, int skip) { *ticket = skip; }

// Per-trajectory coefficients (fp64 then split to double-float) and a check of
// cu_seqlens: 0 = cu[0] <= cu[1] <= ... <= cu[B] = N.
__device__ __forceinline__ void gae_coef_one(int b, const int32_t *cu, int B, int64_t N, float gamma, float lam,
                                             float lam_c, float alpha, const int *nact, float4 *coef,
                                             unsigned int *err) {
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
__global__ void gae_coef_kernel(const int32_t *cu, int B, int64_t N, float gamma, float lam, float lam_c,
                                float alpha, const int *nact, float4 *coef, unsigned int *err) {
  gae_coef_one(blockIdx.x * blockDim.x + threadIdx.x, cu, B, N, gamma, lam, lam_c, alpha, nact, coef, err);
}
// Both set-up passes in one launch when lambda does not depend on the action
// counts (alpha = 0), one thread per trajectory b: its coefficients and the
// check of cu_seqlens, and the first trajectory of every 1024-token
// sub-chunk that starts inside it (chunk_first[q] = b for cu[b] <= 1024 q <
// cu[b + 1]: with a valid cu_seqlens every sub-chunk is written once).
// chunk_first starts zeroed, so a malformed cu_seqlens (flagged here) still
// leaves every entry a trajectory index.
__global__ void __launch_bounds__(256) gae_prep_kernel(const int32_t *cu, int B, int64_t N, int nsub,
                                                       int *chunk_first, float gamma, float lam, float lam_c,
                                                       float4 *coef, unsigned int *err) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  gae_coef_one(b, cu, B, N, gamma, lam, lam_c, 0.f, nullptr, coef, err);
  seg::chunk_first_of(cu, b, N, nsub, chunk_first);
}

constexpr size_t kScanSmem = kWarpBufBytes * kWarps + 1024;  // + alignment slack

// The scan's shared memory exceeds the default 48 KB: opt in once per kernel
// and device.
sao_status set_scan_smem(void (*kern)(GaeArgs, ScanMaps), int which, int device) {
  constexpr int kMaxDevices = 64;
  static std::once_flag once[4][kMaxDevices];
  static cudaError_t err[4][kMaxDevices];
  if (device < 0 || device >= kMaxDevices) return fail(SAO_ERR_CUDA, "device %d out of range", device);
  std::call_once(once[which][device], [&] {
    err[which][device] = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kScanSmem));
  });
  if (err[which][device] != cudaSuccess)
    return fail(SAO_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err[which][device]));
  return SAO_OK;
}

// One map of a per-token array as [rows][seg] elements, box 32 x 32.
bool scan_map(CUtensorMap *map, const void *ptr, CUtensorMapDataType type, size_t esize, int64_t rows, int seg,
              CUtensorMapSwizzle swizzle) {
  auto fn = tensor_map_encoder();
  if (!fn || (reinterpret_cast<uintptr_t>(ptr) & 15u) != 0) return false;
  cuuint64_t dims[2] = {cuuint64_t(seg), cuuint64_t(rows)};
  cuuint64_t strides[1] = {cuuint64_t(seg) * esize};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, type, 2, const_cast<void *>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The tensor maps of the scan's per-token arrays over their N / seg whole
// lane-segment rows; 0 rows (every piece staged element by element) when an
// array is not 16-byte aligned or there is not one whole chunk.
int64_t scan_maps(const float *values, const uint8_t *m, const float *adv, const float *ret, int64_t N, int seg,
                  ScanMaps *maps) {
  const int64_t rows = N / seg;
  if (rows < 32) return 0;
  const bool ok = scan_map(&maps->v, values, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, rows, seg, CU_TENSOR_MAP_SWIZZLE_128B) &&
                  scan_map(&maps->m, m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, rows, seg, CU_TENSOR_MAP_SWIZZLE_32B) &&
                  scan_map(&maps->adv, adv, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, rows, seg, CU_TENSOR_MAP_SWIZZLE_128B) &&
                  scan_map(&maps->ret, ret, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, rows, seg, CU_TENSOR_MAP_SWIZZLE_128B);
  return ok ? rows : 0;
}

}  // namespace

size_t gae_ws_bytes(int64_t N, int64_t B) {
  const int64_t nchunks = (N + kChunk - 1) / kChunk;
  return round256(sizeof(int)) + round256(sizeof(int) * (B + 1)) +
         round256(sizeof(uint64_t) * kMapWords<true> * nchunks) +
         round256(sizeof(uint64_t) * kStateWords<true> * nchunks) + round256(sizeof(float4) * 2 * (B + 1)) +
         round256(sizeof(int) * (nchunks + 1));
}

sao_status gae_launch(const float *values, const float *rewards, const uint8_t *m, const int32_t *cu,
                      int32_t B, int64_t N, float gamma, float lam, float lam_c, float alpha, float *adv,
                      float *ret, unsigned int *err, void *ws_body, size_t body_bytes, cudaStream_t s) {
  if (N == 0) return SAO_OK;
  // 1024-token sub-chunks (the units of chunk_first and of the count and
  // broadcast passes) and the scan's chunks of 32 lane segments of
  // 32 * pieces tokens: longer segments spread the warp scan and look-back of
  // a chunk over more tokens, as long as the scan keeps enough chunks to
  // share out: 2 pieces from 2^23 tokens (4,096 chunks of 2,048), 4 from 2^25
  // (8,192 of 4,096); measured at 2^23 / 2^24 tokens, 1 piece 49 / 82 us,
  // 2 pieces 39 / 62 us, 4 pieces - / 64 us. Pieces come from N alone, so
  // every device gives the same bits.
  const int64_t nchunks = (N + kChunk - 1) / kChunk;
  if (nchunks > (int64_t(1) << 30)) return fail(SAO_ERR_SHAPE, "too many tokens for the advantage scan");
  const int pieces = N >= (int64_t(1) << 25) ? 4 : (N >= (int64_t(1) << 23) ? 2 : 1);
  const int64_t nscan = (N + int64_t(kChunk) * pieces - 1) / (int64_t(kChunk) * pieces);
  const bool crit_trivial = (gamma == 1.0f && lam_c == 1.0f);
  const size_t map_words = crit_trivial ? kMapWords<false> : kMapWords<true>;
  const size_t state_words = crit_trivial ? kStateWords<false> : kStateWords<true>;
  Carver c(ws_body, body_bytes);
  // ticket, action counts, the publication arrays and chunk_first start at zero
  char *zero_begin = c.base + c.off;
  int *ticket = c.take<int>(1);
  int *nact = c.take<int>(size_t(B) + 1);
  uint64_t *agg = c.take<uint64_t>(map_words * size_t(nscan));
  uint64_t *incl = c.take<uint64_t>(state_words * size_t(nscan));
  int *chunk_first = c.take<int>(size_t(nchunks) + 1);
  char *zero_end = c.base + c.off;
  float4 *coef = c.take<float4>(2 * (size_t(B) + 1));
  if (!c.ok()) return fail(SAO_ERR_WORKSPACE, "workspace too small for the advantage scan");
  SAO_CUDA_TRY(cudaMemsetAsync(zero_begin, 0, size_t(zero_end - zero_begin), s));
  if (const int skip = scan_skip(); skip > 0) {
    preset_ticket_kernel<<<1, 1, 0, s>>>(ticket, skip);
    SAO_CUDA_TRY(cudaGetLastError());
  }
  if (alpha > 0.f) {
    // lambda from each trajectory's action count: chunk_first, the count,
    // then the coefficients
    int slot = launch_begin("gae_chunk_first", s);
    seg::chunk_first_kernel<<<seg::chunk_first_grid(B), 256, 0, s>>>(cu, B, N, int(nchunks), chunk_first);
    SAO_TRY(launch_end(slot, s));
    slot = launch_begin("gae_count", s);
    seg::action_count_kernel<<<seg::action_count_grid(int(nchunks)), 256, 0, s>>>(m, cu, B, N, int(nchunks),
                                                                                    chunk_first, nact);
    SAO_TRY(launch_end(slot, s));
    slot = launch_begin("gae_coef", s);
    gae_coef_kernel<<<(B + 127) / 128, 128, 0, s>>>(cu, B, N, gamma, lam, lam_c, alpha, nact, coef, err);
    SAO_TRY(launch_end(slot, s));
  } else {
    int slot = launch_begin("gae_prep", s);
    gae_prep_kernel<<<(B + 255) / 256, 256, 0, s>>>(cu, B, N, int(nchunks), chunk_first, gamma, lam, lam_c, coef,
                                                    err);
    SAO_TRY(launch_end(slot, s));
  }
  if (gamma == 1.0f && lam == 1.0f && lam_c == 1.0f && !(alpha > 0.f)) {
    // gamma = lambda = 1: every delta telescopes, A = R_b - V on the action
    // tokens and the return is R_b, exactly what the scan would produce (its
    // double-float lambda-return is R_b itself): one streaming pass, after
    // the set-up kernel's check of cu_seqlens
    int slot = launch_begin("gae_telescoped", s);
    seg::traj_broadcast_kernel<true><<<seg::broadcast_grid(int(nchunks)), 256, 0, s>>>(
        rewards, m, cu, B, N, int(nchunks), chunk_first, adv, values, ret);
    return launch_end(slot, s);
  }
  GaeArgs a;
  a.values = values;
  a.rewards = rewards;
  a.m = m;
  a.cu = cu;
  a.B = B;
  a.N = N;
  a.nchunks = int(nscan);
  a.pieces = pieces;
  a.nsub = int(nchunks);
  a.coef = coef;
  a.chunk_first = chunk_first;
  a.ticket = ticket;
  a.agg = agg;
  a.incl = incl;
  a.adv = adv;
  a.ret = ret;
  a.err = err;
  a.wait_ns = scan_wait_ns();
  ScanMaps maps;
  a.tma_rows = scan_maps(values, m, adv, ret, N, 32 * pieces, &maps);
  DeviceInfo di;
  SAO_TRY(device_info(&di));
  // segments of 1 or 2 pieces: two chunks in flight per warp
  const bool pipe = pieces <= kMaxPieces / 2;
  auto kern = crit_trivial ? (pipe ? gae_scan_kernel<false, true> : gae_scan_kernel<false, false>)
                           : (pipe ? gae_scan_kernel<true, true> : gae_scan_kernel<true, false>);
  SAO_TRY(set_scan_smem(kern, (crit_trivial ? 0 : 2) + (pipe ? 1 : 0), di.device));
  // persistent: as many warps as fit on the GPU, never more than chunks
  const int64_t ctas = (nscan + kWarps - 1) / kWarps;
  const int64_t resident = int64_t(di.sm_count) * kMinBlocks;
  const unsigned grid = unsigned(ctas < resident ? ctas : resident);
  int slot = launch_begin("gae_scan", s);
  kern<<<grid, kThreads, kScanSmem, s>>>(a, maps);
  return launch_end(slot, s);
}

}  // namespace sao
