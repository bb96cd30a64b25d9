// Scoring pass: per-token sums for the Renyi-2 entropy (Eq. 3-4) and the
// consistency signal (Eq. 6) in one read of x, x', x''.
//
// One warp per row; lane l reads 16-byte chunks l, l+32, l+64, ... of each of
// the three streams (fully coalesced 512-byte warp requests), a batch of
// chunks per stream in flight before any arithmetic; bf16, fp16 or fp32.  Each chunk's partial
// sums of |x|, x^2, x'^2, x''^2 come from a depth-3 fp32 tree; the partials
// are accumulated error-free as double-floats (TwoSum), so every sum carries
// at most score_depth() roundings whatever D is.  P = x'.x'' is accumulated
// error-free term by term, since the ordering by s needs it to far better
// than fp32.  16-bit chunks are processed two at a time with the packed f32x2
// instructions (half the issue slots; each half rounds exactly like the
// scalar operation), so each lane carries two double-float accumulators per
// sum, one for its even-numbered chunks and one for its odd ones.  The
// epilogue derives the fp32 selection keys from the unrounded double-float
// sums (double-float arithmetic, one final rounding), all without fp64
// (GB300's fp64 rate would stall the warp).
#pragma once

#include <cmath>

#include "tr_df.cuh"
#include "tr_internal.cuh"
#include "tr_record.cuh"

namespace tr {
namespace {

__device__ __forceinline__ uint4 ld_stream(const uint4 *p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

// ---- packed pairs: two fp32 values in one 64-bit register pair, operated on
// by the f32x2 instructions (one issue slot for both halves, each half
// rounded to nearest exactly like its scalar counterpart).
__device__ __forceinline__ uint64_t pk(uint32_t lo, uint32_t hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ void unpk(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t sub2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

// A pair of double-float accumulators (one per half).
struct DF2 {
  uint64_t hi, lo;
};
__device__ __forceinline__ void df2_add(DF2 &a, uint64_t v) {  // TwoSum per half
  const uint64_t t = add2(a.hi, v);
  const uint64_t bb = sub2(t, a.hi);
  const uint64_t aa = sub2(t, bb);
  a.lo = add2(a.lo, add2(sub2(a.hi, aa), sub2(v, bb)));
  a.hi = t;
}
// Folds the two halves into one double-float accumulator.
__device__ __forceinline__ DF df2_fold(const DF2 &a) {
  float h0, h1, l0, l1;
  unpk(a.hi, h0, h1);
  unpk(a.lo, l0, l1);
  DF r{h0, l0};
  df_merge(r, h1, l1);
  return r;
}

struct Acc2 {
  DF2 l1, s2, a, b, p;
};

// fp32 bit patterns of the two 16-bit elements of word w (low half first):
// bf16 by shifting, fp16 by exact conversion (subnormals included).
template <int kDt>
__device__ __forceinline__ void halves(uint32_t w, uint32_t &lo, uint32_t &hi) {
  if (kDt == TR_BF16) {
    lo = w << 16;
    hi = w & 0xffff0000u;
  } else {
    float flo, fhi;
    asm("{\n .reg .f16 l, h;\n mov.b32 {l, h}, %2;\n cvt.f32.f16 %0, l;\n cvt.f32.f16 %1, h;\n}"
        : "=f"(flo), "=f"(fhi)
        : "r"(w));
    lo = __float_as_uint(flo);
    hi = __float_as_uint(fhi);
  }
}

// Two 16-byte chunks (u, v) of 16-bit elements (bf16 or fp16) of each stream
// at once: half 0 of every packed value belongs to chunk u, half 1 to chunk
// v.  Per chunk: depth-3 trees of |x|, x^2, x'^2, x''^2 (squares and products
// of bf16 or fp16 values are exact in fp32, so only the additions round; x^2
// is taken as |x|^2, the same value) and the eight exact products x'x''
// through TwoSum one by one.  Chunk u's terms enter accumulator half 0,
// chunk v's half 1.
template <int kDt>
__device__ __forceinline__ void chunk2_half(const uint4 &xu, const uint4 &xv, const uint4 &pu, const uint4 &pv,
                                            const uint4 &qu, const uint4 &qv, Acc2 &acc) {
  const uint32_t wxu[4] = {xu.x, xu.y, xu.z, xu.w}, wxv[4] = {xv.x, xv.y, xv.z, xv.w};
  const uint32_t wpu[4] = {pu.x, pu.y, pu.z, pu.w}, wpv[4] = {pv.x, pv.y, pv.z, pv.w};
  const uint32_t wqu[4] = {qu.x, qu.y, qu.z, qu.w}, wqv[4] = {qv.x, qv.y, qv.z, qv.w};
  uint64_t l[4], s[4], a[4], b[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint32_t x0u, x1u, x0v, x1v, p0u, p1u, p0v, p1v, q0u, q1u, q0v, q1v;
    halves<kDt>(wxu[i] & 0x7fff7fffu, x0u, x1u);  // |x|: both formats keep the sign in bit 15
    halves<kDt>(wxv[i] & 0x7fff7fffu, x0v, x1v);
    halves<kDt>(wpu[i], p0u, p1u);
    halves<kDt>(wpv[i], p0v, p1v);
    halves<kDt>(wqu[i], q0u, q1u);
    halves<kDt>(wqv[i], q0v, q1v);
    const uint64_t x0 = pk(x0u, x0v), x1 = pk(x1u, x1v);
    const uint64_t p0 = pk(p0u, p0v), p1 = pk(p1u, p1v);
    const uint64_t q0 = pk(q0u, q0v), q1 = pk(q1u, q1v);
    l[i] = add2(x0, x1);
    s[i] = fma2(x0, x0, mul2(x1, x1));
    a[i] = fma2(p0, p0, mul2(p1, p1));
    b[i] = fma2(q0, q0, mul2(q1, q1));
    df2_add(acc.p, mul2(p0, q0));
    df2_add(acc.p, mul2(p1, q1));
  }
  df2_add(acc.l1, add2(add2(l[0], l[1]), add2(l[2], l[3])));
  df2_add(acc.s2, add2(add2(s[0], s[1]), add2(s[2], s[3])));
  df2_add(acc.a, add2(add2(a[0], a[1]), add2(a[2], a[3])));
  df2_add(acc.b, add2(add2(b[0], b[1]), add2(b[2], b[3])));
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

// Warp-wide reduction of one row's partial sums and the row's outputs: the
// five sums, the fp32 selection keys, and optionally H2 and s.  Lane 0 writes.
__device__ __forceinline__ void finish_row(Acc &acc, long long row, float4 *__restrict__ stats,
                                           float *__restrict__ h2, float *__restrict__ s_out, int lane) {
  df_warp_sum(acc.l1);
  df_warp_sum(acc.s2);
  df_warp_sum(acc.a);
  df_warp_sum(acc.b);
  df_warp_sum(acc.p);
  if (lane == 0) write_record(acc, row, stats, h2, s_out);
}

// One round: lane l takes chunks base + l + 32u (u < kB) of each stream,
// all loads issued before any arithmetic; with kGuard, chunks at or past c1
// are zeros (which add nothing).
template <int kDt, int kB, bool kGuard>
__device__ __forceinline__ void accumulate_round(const uint4 *__restrict__ rx, const uint4 *__restrict__ rp,
                                                 const uint4 *__restrict__ rq, int base, int c1, Acc &acc,
                                                 Acc2 &acc2, int lane) {
  uint4 vx[kB], vp[kB], vq[kB];
#pragma unroll
  for (int u = 0; u < kB; ++u) {
    const int c = base + lane + 32 * u;
    if (!kGuard || c < c1) {
      vx[u] = ld_stream(rx + c);
      vp[u] = ld_stream(rp + c);
      vq[u] = ld_stream(rq + c);
    } else {
      vx[u] = vp[u] = vq[u] = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  if (kDt != TR_F32) {
#pragma unroll
    for (int u = 0; u < kB; u += 2) chunk2_half<kDt>(vx[u], vx[u + 1], vp[u], vp[u + 1], vq[u], vq[u + 1], acc2);
  } else {
#pragma unroll
    for (int u = 0; u < kB; ++u) chunk_f32(vx[u], vp[u], vq[u], acc);
  }
}

// Partial sums of chunks [c0, c1) of one row, read straight from global
// memory in rounds of kB chunks per lane and stream.  When the row's chunks
// are a multiple of 32 (every lane has the same count) the last round is cut
// to the chunks that remain (6, 4 or 2 per lane, fewer than a full round), so
// no lane works on padding.
template <int kDt>
__device__ __forceinline__ void accumulate_global(const uint4 *__restrict__ rx, const uint4 *__restrict__ rp,
                                                  const uint4 *__restrict__ rq, int c0, int c1, Acc &acc,
                                                  int lane) {
  constexpr int kB = kDt != TR_F32 ? kScoreBatchBf16 : kScoreBatchF32;
  static_assert(kB % 2 == 0, "bf16 chunks are summed in pairs");
  Acc2 acc2{};
  int base = c0;
  for (; base + 32 * kB <= c1; base += 32 * kB) accumulate_round<kDt, kB, false>(rx, rp, rq, base, c1, acc, acc2, lane);
  const int rest = c1 - base;
  if (rest > 0) {
    if (kB > 6 && rest == 32 * 6)
      accumulate_round<kDt, 6, false>(rx, rp, rq, base, c1, acc, acc2, lane);
    else if (kB > 4 && rest == 32 * 4)
      accumulate_round<kDt, 4, false>(rx, rp, rq, base, c1, acc, acc2, lane);
    else if (rest == 32 * 2)
      accumulate_round<kDt, 2, false>(rx, rp, rq, base, c1, acc, acc2, lane);
    else
      accumulate_round<kDt, kB, true>(rx, rp, rq, base, c1, acc, acc2, lane);
  }
  if (kDt != TR_F32) {
    // Half 0 holds this lane's even-numbered chunks, half 1 its odd ones.
    const DF l1 = df2_fold(acc2.l1), s2 = df2_fold(acc2.s2), a = df2_fold(acc2.a), b = df2_fold(acc2.b),
             p = df2_fold(acc2.p);
    df_merge(acc.l1, l1.hi, l1.lo);
    df_merge(acc.s2, s2.hi, s2.lo);
    df_merge(acc.a, a.hi, a.lo);
    df_merge(acc.b, b.hi, b.lo);
    df_merge(acc.p, p.hi, p.lo);
  }
}

// Scores one row (one warp) straight from global memory.
template <int kDt>
__device__ __forceinline__ void score_row(const uint4 *__restrict__ x, const uint4 *__restrict__ xp,
                                          const uint4 *__restrict__ xq, int nchunks, long long row,
                                          float4 *__restrict__ stats, float *__restrict__ h2,
                                          float *__restrict__ s_out, int lane) {
  Acc acc{{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
  accumulate_global<kDt>(x + row * nchunks, xp + row * nchunks, xq + row * nchunks, 0, nchunks, acc, lane);
  finish_row(acc, row, stats, h2, s_out, lane);
}

}  // namespace
}  // namespace tr
