// Scoring pass: per-token sums for the Renyi-2 entropy (Eq. 3-4) and the
// consistency signal (Eq. 6) in one read of x, x', x''.
//
// One warp per row; lane l reads 16-byte chunks l, l+32, l+64, ... of each of
// the three streams (fully coalesced 512-byte warp requests), kScoreBatch
// chunks per stream in flight before any arithmetic.  Each chunk's partial
// sums of |x|, x^2, x'^2, x''^2 come from a depth-3 fp32 tree; the partials
// are accumulated error-free as double-floats (TwoSum), so every sum carries
// at most score_depth() roundings whatever D is.  P = x'.x'' is accumulated
// error-free term by term, since the ordering by s needs it to far better
// than fp32.  The epilogue derives the fp32 selection keys from the
// unrounded double-float sums (double-float arithmetic, one final rounding),
// all without fp64 (GB300's fp64 rate would stall the warp).
#pragma once

#include <cmath>

#include "tr_df.cuh"
#include "tr_internal.cuh"

namespace tr {
namespace {

__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

// Error-free sum: s + e = a + b exactly (Knuth's TwoSum, no ordering assumption).
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
  s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float aa = __fsub_rn(s, bb);
  e = __fadd_rn(__fsub_rn(a, aa), __fsub_rn(b, bb));
}

__device__ __forceinline__ float lo_bf16(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_bf16(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

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

// Eight bf16 elements of each stream: depth-3 trees for |x|, x^2, x'^2, x''^2
// (bf16 squares are exact in fp32, so only the additions round); the eight
// exact products x'x'' go through TwoSum one by one.
__device__ __forceinline__ void chunk_bf16(const uint4 &vx, const uint4 &vp, const uint4 &vq, Acc &acc) {
  const uint32_t wx[4] = {vx.x, vx.y, vx.z, vx.w};
  const uint32_t wp[4] = {vp.x, vp.y, vp.z, vp.w};
  const uint32_t wq[4] = {vq.x, vq.y, vq.z, vq.w};
  float l[4], s[4], a[4], b[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float x0 = lo_bf16(wx[i]), x1 = hi_bf16(wx[i]);
    const float p0 = lo_bf16(wp[i]), p1 = hi_bf16(wp[i]);
    const float q0 = lo_bf16(wq[i]), q1 = hi_bf16(wq[i]);
    l[i] = fabsf(x0) + fabsf(x1);
    s[i] = fmaf(x0, x0, x1 * x1);
    a[i] = fmaf(p0, p0, p1 * p1);
    b[i] = fmaf(q0, q0, q1 * q1);
    df_add(acc.p, p0 * q0);
    df_add(acc.p, p1 * q1);
  }
  df_add(acc.l1, (l[0] + l[1]) + (l[2] + l[3]));
  df_add(acc.s2, (s[0] + s[1]) + (s[2] + s[3]));
  df_add(acc.a, (a[0] + a[1]) + (a[2] + a[3]));
  df_add(acc.b, (b[0] + b[1]) + (b[2] + b[3]));
}

// Four fp32 elements of each stream: depth-2 trees (plus the rounding of each
// square); products split exactly into p + pe with an FMA, both enter P.
__device__ __forceinline__ void chunk_f32(const uint4 &vx, const uint4 &vp, const uint4 &vq, Acc &acc) {
  const float x[4] = {__uint_as_float(vx.x), __uint_as_float(vx.y), __uint_as_float(vx.z), __uint_as_float(vx.w)};
  const float p[4] = {__uint_as_float(vp.x), __uint_as_float(vp.y), __uint_as_float(vp.z), __uint_as_float(vp.w)};
  const float q[4] = {__uint_as_float(vq.x), __uint_as_float(vq.y), __uint_as_float(vq.z), __uint_as_float(vq.w)};
  df_add(acc.l1, (fabsf(x[0]) + fabsf(x[1])) + (fabsf(x[2]) + fabsf(x[3])));
  df_add(acc.s2, fmaf(x[0], x[0], x[1] * x[1]) + fmaf(x[2], x[2], x[3] * x[3]));
  df_add(acc.a, fmaf(p[0], p[0], p[1] * p[1]) + fmaf(p[2], p[2], p[3] * p[3]));
  df_add(acc.b, fmaf(q[0], q[0], q[1] * q[1]) + fmaf(q[2], q[2], q[3] * q[3]));
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float pr = p[i] * q[i];
    const float pe = fmaf(p[i], q[i], -pr);
    df_add(acc.p, pr);
    acc.p.lo += pe;
  }
}

__device__ __forceinline__ void df_warp_sum(DF &v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float oh = __shfl_xor_sync(0xffffffffu, v.hi, o);
    const float ol = __shfl_xor_sync(0xffffffffu, v.lo, o);
    df_merge(v, oh, ol);
  }
}

// Scores one row (one warp): the five sums, the fp32 selection keys, and
// optionally H2 and s.
template <bool kBf16>
__device__ __forceinline__ void score_row(const uint4 *__restrict__ x, const uint4 *__restrict__ xp,
                                          const uint4 *__restrict__ xq, int nchunks, long long row,
                                          float4 *__restrict__ stats, float *__restrict__ h2,
                                          float *__restrict__ s_out, int lane) {
  const uint4 *rx = x + row * nchunks;
  const uint4 *rp = xp + row * nchunks;
  const uint4 *rq = xq + row * nchunks;
  Acc acc{{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
  for (int c0 = lane; c0 < nchunks; c0 += 32 * kScoreBatch) {
    uint4 vx[kScoreBatch], vp[kScoreBatch], vq[kScoreBatch];
#pragma unroll
    for (int u = 0; u < kScoreBatch; ++u) {
      const int c = c0 + 32 * u;
      if (c < nchunks) {
        vx[u] = ld_stream(rx + c);
        vp[u] = ld_stream(rp + c);
        vq[u] = ld_stream(rq + c);
      } else {
        vx[u] = vp[u] = vq[u] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int u = 0; u < kScoreBatch; ++u) {
      if (kBf16)
        chunk_bf16(vx[u], vp[u], vq[u], acc);
      else
        chunk_f32(vx[u], vp[u], vq[u], acc);
    }
  }
  df_warp_sum(acc.l1);
  df_warp_sum(acc.s2);
  df_warp_sum(acc.a);
  df_warp_sum(acc.b);
  df_warp_sum(acc.p);
  if (lane == 0) {
    const df::F2 L1 = df::fast_two_sum(acc.l1.hi, acc.l1.lo), S2 = df::fast_two_sum(acc.s2.hi, acc.s2.lo);
    const df::F2 A = df::fast_two_sum(acc.a.hi, acc.a.lo), B = df::fast_two_sum(acc.b.hi, acc.b.lo);
    const df::F2 P = df::two_sum(acc.p.hi, acc.p.lo);
    const float l1 = df::round(L1), s2 = df::round(S2), sa = df::round(A), sb = df::round(B);
    const float ph = P.h, pl = P.l;
    // Selection keys: R = L1^2 / S2 (H2 = log R, Eq. 3-4) and
    // s = P / (sqrt(A) sqrt(B)) (Eq. 6), evaluated in double-float from the
    // unrounded sums and rounded once to fp32.  NaN marks a row whose sums
    // left the fp32 error model (non-finite, overflowed or underflowed): the
    // selection recomputes it exactly.
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
}

}  // namespace
}  // namespace tr
