// Double-float arithmetic on fp32 pairs (about 48 significant bits) from
// error-free transformations (Knuth's two-sum, Dekker's fast two-sum, the
// fused multiply-add's exact product remainder), for the per-trajectory
// epilogues that would otherwise need the fp64 pipe, which is narrow on
// GB300.
#pragma once

#include <cuda_runtime.h>

namespace sao {
namespace dfl {

struct F2 {
  float hi, lo;
};

__device__ __forceinline__ F2 quick_two_sum(float a, float b) {  // |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ F2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}
// A pair whose low part may have grown (a compensated sum), renormalised.
__device__ __forceinline__ F2 norm(float hi, float lo) { return two_sum(hi, lo); }
__device__ __forceinline__ F2 add(F2 x, F2 y) {
  const F2 s = two_sum(x.hi, y.hi);
  return quick_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(x.lo, y.lo)));
}
__device__ __forceinline__ F2 neg(F2 x) { return {-x.hi, -x.lo}; }
__device__ __forceinline__ F2 sub(F2 x, F2 y) { return add(x, neg(y)); }
__device__ __forceinline__ F2 mul(F2 x, F2 y) {
  const float p = __fmul_rn(x.hi, y.hi);
  float e = __fmaf_rn(x.hi, y.hi, -p);
  e = __fmaf_rn(x.hi, y.lo, e);
  e = __fmaf_rn(x.lo, y.hi, e);
  return quick_two_sum(p, e);
}
// x / n for a positive integer n below 2^24 (exact as a float): the first
// quotient's remainder x.hi - q1 n is exact in one fused multiply-add, so a
// second quotient corrects it.
__device__ __forceinline__ F2 div_int(F2 x, int n) {
  const float d = float(n);
  const float q1 = __fdiv_rn(x.hi, d);
  const float r = __fadd_rn(__fmaf_rn(-q1, d, x.hi), x.lo);
  return quick_two_sum(q1, __fdiv_rn(r, d));
}
__device__ __forceinline__ float round(F2 x) { return __fadd_rn(x.hi, x.lo); }

}  // namespace dfl
}  // namespace sao
