// Double-float arithmetic on fp32 hardware (a value is hi + lo, |lo| <= ulp(hi)/2):
// the classic error-free transformations TwoSum, FastTwoSum and TwoProd (via
// FMA) and the double-float product, quotient and square root built on them.
// Each of mul/div/sqrt is accurate to a few u^2 relative (u = 2^-24) as long
// as no intermediate underflows or overflows, far below what one final
// rounding to fp32 adds.  fp64 is avoided on purpose: GB300's fp64 rate is a
// small fraction of its fp32 rate.
#pragma once

namespace tr {
namespace df {

struct F2 {
  float h, l;
};

// s + e == a + b exactly, any magnitudes.
__device__ __forceinline__ F2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float aa = __fsub_rn(s, bb);
  return F2{s, __fadd_rn(__fsub_rn(a, aa), __fsub_rn(b, bb))};
}
// s + e == a + b exactly when |a| >= |b|.
__device__ __forceinline__ F2 fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return F2{s, __fsub_rn(b, __fsub_rn(s, a))};
}
// p + e == a * b exactly.
__device__ __forceinline__ F2 two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return F2{p, __fmaf_rn(a, b, -p)};
}
__device__ __forceinline__ F2 mul(const F2 &x, const F2 &y) {
  const F2 p = two_prod(x.h, y.h);
  return fast_two_sum(p.h, __fmaf_rn(x.h, y.l, __fmaf_rn(x.l, y.h, p.l)));
}
__device__ __forceinline__ F2 div(const F2 &a, const F2 &b) {
  const float q1 = __fdiv_rn(a.h, b.h);
  const F2 t = two_prod(q1, b.h);
  const float r = __fsub_rn(__fadd_rn(__fsub_rn(__fsub_rn(a.h, t.h), t.l), a.l), __fmul_rn(q1, b.l));
  return fast_two_sum(q1, __fdiv_rn(r, b.h));
}
__device__ __forceinline__ F2 sqrt(const F2 &a) {
  const float s = __fsqrt_rn(a.h);
  const F2 p = two_prod(s, s);
  const float r = __fadd_rn(__fsub_rn(__fsub_rn(a.h, p.h), p.l), a.l);
  return fast_two_sum(s, __fdiv_rn(r, __fmul_rn(2.f, s)));
}
__device__ __forceinline__ float round(const F2 &x) { return __fadd_rn(x.h, x.l); }

}  // namespace df
}  // namespace tr
