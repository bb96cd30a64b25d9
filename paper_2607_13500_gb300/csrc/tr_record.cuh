// The per-row statistics record that the selection reads (include/tr.h,
// tr_score): the five sums of Eq. 3-4 and Eq. 6 accumulated as double-floats,
// and the record written from them.  Two producers share it: the scoring
// pass (k_score) and the encoder-MLP GEMM whose epilogue scores the rows it
// produces (k_mlp_gemm).
#pragma once

#include <cmath>

#include "tr_df.cuh"
#include "tr_internal.cuh"

namespace tr {
namespace {

// Error-free sum: s + e = a + b exactly (Knuth's TwoSum, no ordering assumption).
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
  s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float aa = __fsub_rn(s, bb);
  e = __fadd_rn(__fsub_rn(a, aa), __fsub_rn(b, bb));
}


// Double-float accumulator: hi + lo carries the sum, hi exact in TwoSum.
struct DF {
  float hi, lo;
};
__device__ __forceinline__ void df_add(DF &a, float v) {
  float t, e;
  two_sum(a.hi, v, t, e);
  a.hi = t;
  a.lo += e;
}
__device__ __forceinline__ void df_merge(DF &a, float hi, float lo) {
  float t, e;
  two_sum(a.hi, hi, t, e);
  a.hi = t;
  a.lo = a.lo + lo + e;
}

struct Acc {
  DF l1, s2, a, b, p;
};

// Writes row `row`'s record from its double-float sums: [0..3] L1, S2, A, B
// rounded to fp32, [4..5] P as hi + lo, [6] the importance key R = L1^2 / S2
// (H2 = log R, Eq. 3-4) and [7] the consistency key s = P / (sqrt(A) sqrt(B))
// (Eq. 6), both evaluated in double-float from the unrounded sums and rounded
// once to fp32.  NaN keys mark a row whose sums left the fp32 error model
// (non-finite, overflowed or underflowed): the selection recomputes it
// exactly.  Optional H2 and s outputs.
__device__ __forceinline__ void write_record(const Acc &acc, long long row, float4 *__restrict__ stats,
                                             float *__restrict__ h2, float *__restrict__ s_out) {
  const df::F2 L1 = df::fast_two_sum(acc.l1.hi, acc.l1.lo), S2 = df::fast_two_sum(acc.s2.hi, acc.s2.lo);
  const df::F2 A = df::fast_two_sum(acc.a.hi, acc.a.lo), B = df::fast_two_sum(acc.b.hi, acc.b.lo);
  const df::F2 P = df::two_sum(acc.p.hi, acc.p.lo);
  const float l1 = df::round(L1), s2 = df::round(S2), sa = df::round(A), sb = df::round(B);
  const float ph = P.h, pl = P.l;
  const bool bad_r = !(isfinite(l1) && isfinite(s2)) || (l1 != 0.f && (s2 < kTiny || s2 > kHuge));
  const bool bad_s = !(isfinite(sa) && isfinite(sb) && isfinite(ph) && isfinite(pl)) || sa < kTiny ||
                     sb < kTiny || sa > kHuge || sb > kHuge;
  const float nan = __int_as_float(0x7fc00000);
  float r = nan, sv = nan;
  if (!bad_r) r = l1 == 0.f ? 1.f : df::round(df::div(df::mul(L1, L1), S2));
  if (!bad_s) sv = df::round(df::div(P, df::mul(df::sqrt(A), df::sqrt(B))));
  stats[2 * row] = make_float4(l1, s2, sa, sb);
  stats[2 * row + 1] = make_float4(ph, pl, r, sv);
  if (h2) h2[row] = l1 > 0.f ? logf(r) : 0.f;
  if (s_out) s_out[row] = (sa > 0.f && sb > 0.f) ? sv : 0.f;
}

}  // namespace
}  // namespace tr
