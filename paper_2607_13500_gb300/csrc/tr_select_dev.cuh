// Selection of Algorithm 1 (Stage I top-K1 by H2, Stage II ascending sort by s
// and stride pick), one CTA per image, with exact decisions.
//
// Keys.  H2 = log R with R = L1^2 / S2 (Eq. 3-4: sum_j p_j^2 = S2 / L1^2),
// so ranking by H2 is ranking by R; s = P / sqrt(A B) (Eq. 6).  The score
// pass leaves fp32 keys R32 and s32 in each row's statistics record.  Stage
// I finds the K1-th key by a radix select and needs an order only near an
// uncertain cut; Stage II sorts X_rem by s (keys packed with the token index
// into 64-bit words: a register bitonic sort up to 512 rows, else value
// buckets ranked per row, and where the values crowd a register bitonic sort
// up to 2048 rows, a stratified sample sort or a stable radix sort), so that
// equal keys order by the lower index.
//
// Certification.  The score pass's sums carry proven error bounds (Bounds),
// so a cut between sorted neighbours is certain when their key intervals do
// not overlap; with a uniform relative (R) or monotone absolute (s) bound it
// suffices to test adjacent pairs.  Only decisions matter: the cut at K1 for
// Stage I and the neighbourhood of each stride position for Stage II.  The
// tokens of an uncertain run (a maximal stretch of uncertain cuts around a
// decision) are recomputed in double-float from error-free sums first; when
// those keys separate every pair of the run (any run that is not an exact
// tie, in practice) they rank it.  Otherwise the run is recomputed exactly
// -- its five sums as integers, from the input bits -- and ranked by exact
// rational comparison (cross products of big integers), ties to the lower
// index.  Rows whose fp32 sums left the error model (non-finite, overflowed,
// tiny) are recomputed exactly up front.
#pragma once

#include <cfloat>
#include <climits>
#include <cmath>

#include "tr_df.cuh"
#include "tr_internal.cuh"

namespace tr {
namespace {

enum : uint8_t {
  F_IMP = 1,     // in X_imp
  F_DIV = 2,     // in X_div
  F_XL = 4,      // exact L1, S2 in the row's ExactRec
  F_XS = 8,      // exact P, A, B in the row's ExactRec
  F_NEEDL = 16,  // exact L1, S2 requested
  F_NEEDS = 32,  // exact P, A, B requested
  F_RUN = 64,    // lies in an uncertain run around a stride position
  F_DF = 128,    // with F_NEED*: the double-float tier may settle it; alone: it did
                 // (the row's ExactRec holds the current stage's double-float key)
};

// ---------------------------------------------------------------- float keys
__device__ __forceinline__ uint32_t ord32(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unord32(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
// fp32 keys from the statistics record; NaN = outside the fp32 error model.
__device__ __forceinline__ float key_r(const float *st) { return __ldcg(st + 6); }
__device__ __forceinline__ float key_s(const float *st) { return __ldcg(st + 7); }
// Both keys in one 8-byte load (records are 32-byte aligned).
__device__ __forceinline__ float2 key_rs(const float *st) { return __ldcg(reinterpret_cast<const float2 *>(st + 6)); }
constexpr int kKeyIlp = 4;  // rows whose keys a thread loads before it uses any

// ---- a Big truncated to a 64-bit mantissa: value in [m 2^e, (m + 1) 2^e) ----
// Integer-only (the GPU's fp64 rate is far too low for this path).
struct Fx {
  unsigned long long m;  // top bit set, or 0 for the value 0
  int e;
};
__device__ __forceinline__ Fx big_fx(const Big &b) {
  if (b.n == 0) return Fx{0ull, 0};
  const int n = b.n;
  const unsigned long long top = ((unsigned long long)b.l[n - 1] << 32) | (n >= 2 ? b.l[n - 2] : 0u);
  const uint32_t third = n >= 3 ? b.l[n - 3] : 0u;
  const int z = __clzll(top);  // < 32: the top limb is non-zero
  const unsigned long long m = z ? (top << z) | ((unsigned long long)third >> (32 - z)) : top;
  return Fx{m, 32 * (b.e + n - 2) - z};
}
__device__ __forceinline__ Fx fx_one() { return Fx{1ull << 63, -63}; }
// Product truncated to 64 bits (relative error below 2^-63).
__device__ __forceinline__ Fx fx_mul(const Fx &a, const Fx &b) {
  if (!a.m || !b.m) return Fx{0ull, 0};
  const unsigned long long hi = __umul64hi(a.m, b.m), lo = a.m * b.m;
  if (hi >> 63) return Fx{hi, a.e + b.e + 64};
  return Fx{(hi << 1) | (lo >> 63), a.e + b.e + 63};
}
// sign(x - y) when |x - y| exceeds 2^-57 of max(x, y), else 0 (too close to
// call: each side is a product of at most four truncated factors, within
// 2^-60 of its value).
__device__ __forceinline__ int fx_cmp(const Fx &x, const Fx &y) {
  if (!x.m || !y.m) return (x.m != 0) - (y.m != 0);
  const bool xbig = x.e >= y.e;
  const Fx &b = xbig ? x : y, &s = xbig ? y : x;
  const int sh = b.e - s.e;
  const unsigned long long sm = sh >= 64 ? 0ull : s.m >> sh;
  if (b.m > sm && b.m - sm > 128ull) return xbig ? 1 : -1;
  if (sm > b.m && sm - b.m > 128ull) return xbig ? -1 : 1;
  return 0;
}
// Mantissa of a non-zero Fx as a float in [1, 2], rounded to nearest: the Fx
// value is fx_mant(x) * 2^(x.e + 63).
__device__ __forceinline__ float fx_mant(const Fx &x) { return __ull2float_rn(x.m) * 0x1p-63f; }
__device__ __forceinline__ float fx_log(const Fx &x) {  // natural log of a non-zero Fx
  return logf(fx_mant(x)) + (float)(x.e + 63) * 0.69314718f;
}

// The mantissa of a non-zero Fx as a double-float in [1, 2] (within 2^-47):
// the Fx value is fx_f2(x) * 2^(x.e + 63).
__device__ __forceinline__ df::F2 fx_f2(const Fx &x) {
  const float h = (float)(x.m >> 40) * 0x1p40f;             // top 24 bits, exact
  const float l = __ull2float_rn(x.m & ((1ull << 40) - 1));  // the rest, rounded
  const df::F2 v = df::fast_two_sum(h, l);
  return df::F2{v.h * 0x1p-63f, v.l * 0x1p-63f};
}

// Keys of a row settled exactly: the same double-float evaluation as the
// score pass, from the exact sums (truncated to 64 bits), rounded once.
// Out of line, like every path that only near-ties and extreme rows take:
// the select kernel is bound by instruction fetch, so the common path's
// code is kept compact.
__device__ __noinline__ float exact_r_key(const ExactRec &r) {
  if (r.flags_l & kRecNonFiniteX) return 0.f;
  if (r.l1.n == 0) return 1.f;
  const Fx l1 = big_fx(r.l1), s2 = big_fx(r.s2);
  const df::F2 L = fx_f2(l1), S = fx_f2(s2);
  return ldexpf(df::round(df::div(df::mul(L, L), S)), 2 * (l1.e + 63) - (s2.e + 63));
}
__device__ __noinline__ float exact_h2(const ExactRec &r) {
  if (r.flags_l & kRecNonFiniteX) return -INFINITY;
  if (r.l1.n == 0) return 0.f;
  const Fx l1 = big_fx(r.l1), s2 = big_fx(r.s2);
  return 2.f * fx_log(l1) - fx_log(s2);
}
__device__ __noinline__ float exact_s_key(const ExactRec &r) {
  if (r.flags_s & kRecNonFiniteS) return 2.f;
  if (r.a.n == 0 || r.b.n == 0 || r.p.n == 0) return 0.f;
  const Fx p = big_fx(r.p), a = big_fx(r.a), b = big_fx(r.b);
  // s = P / sqrt(A B); A and B scaled to even exponents so the roots are exact powers of two
  df::F2 A = fx_f2(a), B = fx_f2(b);
  int ea = a.e + 63, eb = b.e + 63;
  if (ea & 1) {
    A = df::F2{A.h * 2.f, A.l * 2.f};
    --ea;
  }
  if (eb & 1) {
    B = df::F2{B.h * 2.f, B.l * 2.f};
    --eb;
  }
  const float v = ldexpf(df::round(df::div(fx_f2(p), df::mul(df::sqrt(A), df::sqrt(B)))), (p.e + 63) - ea / 2 - eb / 2);
  return r.p.neg ? -v : v;
}

// Sorted order: ord[q] is the row at position q, key[row] its 32-bit sort
// key: ~ord32(R32) for the importance order (ascending key = descending R),
// ord32(s32) for the consistency order.
__device__ __forceinline__ float r_of(const uint32_t *key, const uint16_t *ord, int q) {
  return unord32(~key[ord[q]]);
}
__device__ __forceinline__ float s_of(const uint32_t *key, const uint16_t *ord, int q) {
  return unord32(key[ord[q]]);
}

// Cut between importance-sorted positions q-1 and q is certain when the
// smallest R the bounds allow at q-1 exceeds the largest R they allow at q;
// evaluated in fp32 with rounding toward the safe side.
// Certain that a row with key R32 = ra ranks above one with R32 = rb.
__device__ __forceinline__ bool cert_r_val(float ra, float rb, const Bounds &bd) {
  return __fmul_rd(ra, bd.r_lo) > __fmul_ru(rb, bd.r_hi);
}
__device__ __forceinline__ bool cert_r(const uint32_t *key, const uint16_t *ord, int q, const Bounds &bd) {
  return cert_r_val(r_of(key, ord, q - 1), r_of(key, ord, q), bd);
}
// Cut between consistency-sorted positions q-1 and q (ascending s32).
__device__ __forceinline__ bool cert_s(const uint32_t *key, const uint16_t *ord, int q, const Bounds &bd) {
  const float sa = s_of(key, ord, q - 1), sb = s_of(key, ord, q);
  const float hi_a = __fadd_ru(sa, __fmaf_ru(bd.s_rel, fabsf(sa), bd.s_abs));
  const float lo_b = __fsub_rd(sb, __fmaf_ru(bd.s_rel, fabsf(sb), bd.s_abs));
  return lo_b > hi_a;
}

// ---------------------------------------------------------------- exact sums
constexpr int kDig = 20;  // 32-bit digit positions per exact accumulator

struct Term {
  uint32_t m;  // integer significand
  int e;       // value = m * 2^e
  bool nonfinite;
};
// value = m 2^e of element i of a tensor of dtype dt (significand with the
// hidden bit; subnormals use the smallest exponent).
__device__ __forceinline__ Term decode(const void *base, long long i, int dt) {
  Term t;
  if (dt == TR_BF16) {
    const uint32_t b = static_cast<const uint16_t *>(base)[i];
    const uint32_t ex = (b >> 7) & 0xffu, mant = b & 0x7fu;
    t.nonfinite = ex == 0xffu;
    t.m = ex ? (mant | 0x80u) : mant;
    t.e = (ex ? (int)ex : 1) - 134;
  } else if (dt == TR_F16) {
    const uint32_t b = static_cast<const uint16_t *>(base)[i];
    const uint32_t ex = (b >> 10) & 0x1fu, mant = b & 0x3ffu;
    t.nonfinite = ex == 0x1fu;
    t.m = ex ? (mant | 0x400u) : mant;
    t.e = (ex ? (int)ex : 1) - 25;
  } else {
    const uint32_t b = static_cast<const uint32_t *>(base)[i];
    const uint32_t ex = (b >> 23) & 0xffu, mant = b & 0x7fffffu;
    t.nonfinite = ex == 0xffu;
    t.m = ex ? (mant | 0x800000u) : mant;
    t.e = (ex ? (int)ex : 1) - 150;
  }
  return t;
}
__device__ __forceinline__ bool sign_bit(const void *base, long long i, int dt) {
  return dt != TR_F32 ? (static_cast<const uint16_t *>(base)[i] >> 15) != 0
                      : (static_cast<const uint32_t *>(base)[i] >> 31) != 0;
}

// Adds (+/-) m * 2^e into signed 32-bit digit positions relative to 2^base.
__device__ __forceinline__ void add_term(long long *dg, int base, unsigned long long m, int e, bool negative) {
  const int off = e - base;  // >= 0 for every finite input value, see the bases below
  const int k = off >> 5, r = off & 31;
  const unsigned long long lo = m << r;
  const unsigned long long hi = r ? (m >> (64 - r)) : 0ull;
  long long p0 = (long long)(lo & 0xffffffffull), p1 = (long long)(lo >> 32), p2 = (long long)hi;
  if (negative) {
    p0 = -p0;
    p1 = -p1;
    p2 = -p2;
  }
  dg[k] += p0;
  dg[k + 1] += p1;
  if (p2) dg[k + 2] += p2;
}

// Carry-propagates signed digits (value = sum dg[k] 2^(32k + base)) into a
// trimmed sign-magnitude Big.  Returns false when more than kBigLimbs limbs
// would be needed.
//
// The record is built in local storage and written to `out` (global memory)
// with one struct store at the end: every store into an exact record carries
// its final value.  Replica CTAs of one image (k_select_gather) recompute
// the same rows into the same records; a replica that has finished a record
// may already be reading it while another is still writing it, which is
// harmless only because no store ever writes anything but the final bytes.
__device__ bool normalize(const long long *dg, int base, Big &out) {
  uint32_t limb[kDig + 2];
  long long carry = 0;
  for (int k = 0; k < kDig; ++k) {
    const long long t = dg[k] + carry;
    limb[k] = (uint32_t)t;
    carry = t >> 32;
  }
  const bool neg = carry < 0;
  if (neg) {
    carry = 0;
    for (int k = 0; k < kDig; ++k) {
      const long long t = -dg[k] + carry;
      limb[k] = (uint32_t)t;
      carry = t >> 32;
    }
  }
  limb[kDig] = (uint32_t)carry;
  limb[kDig + 1] = (uint32_t)(carry >> 32);
  Big t;
  for (int i = 0; i < kBigLimbs; ++i) t.l[i] = 0u;
  t.n = 0;
  t.e = 0;
  t.neg = 0;
  int hi = kDig + 1;
  while (hi >= 0 && limb[hi] == 0) --hi;
  bool ok = true;
  if (hi >= 0) {
    int lo = 0;
    while (limb[lo] == 0) ++lo;
    const int n = hi - lo + 1;
    if (n > kBigLimbs) {
      ok = false;  // stays the value 0; the caller flags the overflow
    } else {
      for (int i = 0; i < n; ++i) t.l[i] = limb[lo + i];
      t.n = (uint8_t)n;
      t.e = (int16_t)(lo + base / 32);
      t.neg = neg ? 1 : 0;
    }
  }
  out = t;
  return ok;
}

__device__ __forceinline__ void warp_sum_digits(long long *dg) {
  for (int k = 0; k < kDig; ++k) {
    long long v = dg[k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    dg[k] = v;
  }
}

// Exact sums of one row, computed by one warp.  mode 0: L1 = sum|x| and
// S2 = sum x^2; mode 1: A = sum x'^2, B = sum x''^2, P = sum x'x''.
// Digit bases (multiples of 32): |x| has exponent >= -133 (bf16), -24 (fp16)
// or -149 (fp32), products >= -266, -48 or -298; the top digit stays below
// kDig.
__device__ __noinline__ void exact_row(const SelectArgs &a, long long row, int mode, ExactRec *rec, int lane) {
  const int dt = a.dtype;
  const int base1 = -160;
  const int base2 = dt != TR_F32 ? -288 : -320;
  long long d0[kDig], d1[kDig], d2[kDig];
  for (int k = 0; k < kDig; ++k) d0[k] = d1[k] = d2[k] = 0;
  bool nonfinite = false;
  const long long first = row * (long long)a.d;
  if (mode == 0) {
    for (int j = lane; j < a.d; j += 32) {
      const Term t = decode(a.x, first + j, dt);
      if (t.nonfinite) {
        nonfinite = true;
      } else if (t.m) {
        add_term(d0, base1, t.m, t.e, false);
        add_term(d1, base2, (unsigned long long)t.m * t.m, 2 * t.e, false);
      }
    }
  } else {
    const void *xp = a.x_pre ? a.x_pre : a.x;
    for (int j = lane; j < a.d; j += 32) {
      const Term p = decode(xp, first + j, dt);
      const Term q = decode(a.x_post, first + j, dt);
      if (p.nonfinite || q.nonfinite) {
        nonfinite = true;
        continue;
      }
      if (p.m) add_term(d0, base2, (unsigned long long)p.m * p.m, 2 * p.e, false);
      if (q.m) add_term(d1, base2, (unsigned long long)q.m * q.m, 2 * q.e, false);
      if (p.m && q.m) {
        const bool neg = sign_bit(xp, first + j, dt) != sign_bit(a.x_post, first + j, dt);
        add_term(d2, base2, (unsigned long long)p.m * q.m, p.e + q.e, neg);
      }
    }
  }
  nonfinite = __any_sync(0xffffffffu, nonfinite);
  warp_sum_digits(d0);
  warp_sum_digits(d1);
  if (mode == 1) warp_sum_digits(d2);
  if (lane == 0) {
    uint32_t flags = 0;
    if (mode == 0) {
      if (nonfinite) flags |= kRecNonFiniteX;
      bool ok = normalize(d0, base1, rec->l1);
      ok = normalize(d1, base2, rec->s2) && ok;
      if (!ok) flags |= kRecOverflowL;
      rec->flags_l = flags;
    } else {
      if (nonfinite) flags |= kRecNonFiniteS;
      bool ok = normalize(d0, base2, rec->a);
      ok = normalize(d1, base2, rec->b) && ok;
      ok = normalize(d2, base2, rec->p) && ok;
      if (!ok) flags |= kRecOverflowS;
      rec->flags_s = flags;
    }
  }
}

// ---- fast exact sums: one 128-bit integer per sum, in registers ----------
// Every term is m * 2^e with an integer m of at most 2 * kMant bits.  With
// the row's smallest exponent as the base, term m * 2^(e - base) and the sum
// of all d terms fit 127 bits whenever the row's exponent span is moderate
// (always for ordinary activations); the warp checks that first and falls
// back to the digit accumulator above otherwise.
struct Dec {
  uint32_t m;
  int e;
  bool neg, nf;
};
__device__ __forceinline__ Dec dec16(uint32_t h) {
  const uint32_t ex = (h >> 7) & 0xffu, mant = h & 0x7fu;
  return Dec{ex ? (mant | 0x80u) : mant, (ex ? (int)ex : 1) - 134, (h >> 15) != 0, ex == 0xffu};
}
__device__ __forceinline__ Dec dec32(uint32_t b) {
  const uint32_t ex = (b >> 23) & 0xffu, mant = b & 0x7fffffu;
  return Dec{ex ? (mant | 0x800000u) : mant, (ex ? (int)ex : 1) - 150, (b >> 31) != 0, ex == 0xffu};
}

__device__ __forceinline__ Dec dec16h(uint32_t h) {  // IEEE binary16
  const uint32_t ex = (h >> 10) & 0x1fu, mant = h & 0x3ffu;
  return Dec{ex ? (mant | 0x400u) : mant, (ex ? (int)ex : 1) - 25, (h >> 15) != 0, ex == 0x1fu};
}

template <int kDt>
__device__ __forceinline__ void unpack(const uint4 &v, Dec *out) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if (kDt == TR_BF16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i] = dec16(w[i] & 0xffffu);
      out[2 * i + 1] = dec16(w[i] >> 16);
    }
  } else if (kDt == TR_F16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i] = dec16h(w[i] & 0xffffu);
      out[2 * i + 1] = dec16h(w[i] >> 16);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) out[i] = dec32(w[i]);
  }
}

__device__ __forceinline__ void add128(__int128 &acc, unsigned long long m, int sh, bool neg) {
  const __int128 v = (__int128)((unsigned __int128)m << sh);
  acc = neg ? acc - v : acc + v;
}
__device__ __forceinline__ __int128 warp_sum128(__int128 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long lo = __shfl_xor_sync(0xffffffffu, (unsigned long long)v, o);
    const unsigned long long hi = __shfl_xor_sync(0xffffffffu, (unsigned long long)((unsigned __int128)v >> 64), o);
    v += (__int128)(((unsigned __int128)hi << 64) | lo);
  }
  return v;
}

// value = v * 2^base as a trimmed Big (|v| < 2^127, so at most 5 limbs).
// Built in registers (compile-time limb indices, selects instead of an
// indexed array) and stored with one struct write.
__device__ void int128_to_big(__int128 v, int base, Big &out) {
  const bool neg = v < 0;
  const unsigned __int128 mag = neg ? (unsigned __int128)(-v) : (unsigned __int128)v;
  Big t;
#pragma unroll
  for (int i = 0; i < kBigLimbs; ++i) t.l[i] = 0u;
  if (mag == 0) {
    t.n = 0;
    t.e = 0;
    t.neg = 0;
    out = t;
    return;
  }
  const int q = base >> 5, r = base & 31;  // base = 32 q + r, 0 <= r < 32
  const unsigned __int128 lo = mag << r;
  const uint32_t limb[5] = {(uint32_t)lo, (uint32_t)(lo >> 32), (uint32_t)(lo >> 64), (uint32_t)(lo >> 96),
                            r ? (uint32_t)(mag >> (128 - r)) : 0u};
  int first = 4, last = 0;  // lowest and highest non-zero limbs
#pragma unroll
  for (int k = 4; k >= 0; --k)
    if (limb[k]) first = k;
#pragma unroll
  for (int k = 0; k < 5; ++k)
    if (limb[k]) last = k;
#pragma unroll
  for (int i = 0; i < 5; ++i) {
    uint32_t w = 0u;
#pragma unroll
    for (int k = i; k < 5; ++k)
      if (k - i == first) w = limb[k];
    t.l[i] = w;
  }
  t.n = (uint8_t)(last - first + 1);
  t.e = (int16_t)(q + first);
  t.neg = neg ? 1 : 0;
  out = t;
}

// Window for one exact sum: every term and the sum are below 2^top, where
// 2^top exceeds 1.5 x (the fp32 sum of |terms|, itself within 1e-6 of the
// truth); terms are integers times 2^bottom with bottom = top - 126, so the
// signed 128-bit accumulator cannot overflow.  A term with a lower bit below
// 2^bottom does not fit (the row spans > ~95 binades): the caller falls back.
__device__ __forceinline__ int window_bottom(float bound) {
  int ex;
  frexpf(bound * 1.5f, &ex);  // bound * 1.5 < 2^ex
  return ex - 126;
}

constexpr int kWarps = kSelectThreads / 32;

// 128-bit partial sums of the warps, reduced by thread 0.
struct Part128 {
  unsigned long long lo[kWarps * 3], hi[kWarps * 3];
};
__device__ __forceinline__ void part_put(Part128 &p, int slot, __int128 v) {
  p.lo[slot] = (unsigned long long)v;
  p.hi[slot] = (unsigned long long)((unsigned __int128)v >> 64);
}
__device__ __forceinline__ __int128 part_sum(const Part128 &p, int which) {
  __int128 v = 0;
  for (int w = 0; w < kWarps; ++w)
    v += (__int128)(((unsigned __int128)p.hi[w * 3 + which] << 64) | p.lo[w * 3 + which]);
  return v;
}

// A group of warps that works on one row: threads [first, first + size) of
// the CTA, synchronised by named barrier `bar` (1..15; 0 is __syncthreads).
struct Group {
  int first, size, bar;
  __device__ __forceinline__ int tid() const { return (int)threadIdx.x - first; }
  __device__ __forceinline__ void sync() const {
    asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(size) : "memory");
  }
  __device__ __forceinline__ bool all(bool v) const {
    unsigned r;
    asm volatile(
        "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}"
        : "=r"(r)
        : "r"((unsigned)v), "r"(bar), "r"(size)
        : "memory");
    return r != 0;
  }
};

// Exact sums of one row computed by a group of warps (each thread takes
// 16-byte chunks t, t + size, ...), in three 128-bit windows; false
// (uniformly across the group) when a term does not fit its window.
template <int kDt>
__device__ __noinline__ bool exact_row_block(const SelectArgs &a, long long row, int mode, const float *st,
                                             ExactRec *rec, Part128 &part, const Group g) {
  constexpr int kPer = kDt == TR_F32 ? 4 : 8;  // elements per 16-byte chunk
  const int nchunks = a.d / kPer;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  bool fits = true;
  Dec e0[kPer], e1[kPer];
  __int128 s0 = 0, s1 = 0, s2 = 0;
  int b0, b1, b2 = 0;
  if (mode == 0) {
    b0 = window_bottom(__ldcg(st + 0));
    b1 = window_bottom(__ldcg(st + 1));
    const uint4 *px = static_cast<const uint4 *>(a.x) + row * nchunks;
#pragma unroll 4
    for (int c = g.tid(); c < nchunks; c += g.size) {
      unpack<kDt>(__ldg(px + c), e0);
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const Dec &t = e0[i];
        if (!t.m) continue;
        if (t.nf || t.e < b0 || 2 * t.e < b1) {
          fits = false;
          continue;
        }
        add128(s0, t.m, t.e - b0, false);
        add128(s1, (unsigned long long)t.m * t.m, 2 * t.e - b1, false);
      }
    }
  } else {
    const float sa = __ldcg(st + 2), sb = __ldcg(st + 3);
    b0 = window_bottom(sa);
    b1 = window_bottom(sb);
    b2 = window_bottom(__fsqrt_ru(sa) * __fsqrt_ru(sb));
    const uint4 *pp = static_cast<const uint4 *>(a.x_pre ? a.x_pre : a.x) + row * nchunks;
    const uint4 *pq = static_cast<const uint4 *>(a.x_post) + row * nchunks;
#pragma unroll 4
    for (int c = g.tid(); c < nchunks; c += g.size) {
      unpack<kDt>(__ldg(pp + c), e0);
      unpack<kDt>(__ldg(pq + c), e1);
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const Dec &p = e0[i], &q = e1[i];
        if (p.nf || q.nf) {
          fits = false;
          continue;
        }
        if (p.m) {
          if (2 * p.e < b0) fits = false; else add128(s0, (unsigned long long)p.m * p.m, 2 * p.e - b0, false);
        }
        if (q.m) {
          if (2 * q.e < b1) fits = false; else add128(s1, (unsigned long long)q.m * q.m, 2 * q.e - b1, false);
        }
        if (p.m && q.m) {
          if (p.e + q.e < b2) fits = false;
          else add128(s2, (unsigned long long)p.m * q.m, p.e + q.e - b2, p.neg != q.neg);
        }
      }
    }
  }
  if (!g.all(fits)) return false;
  s0 = warp_sum128(s0);
  s1 = warp_sum128(s1);
  s2 = warp_sum128(s2);
  if (lane == 0) {
    part_put(part, warp * 3 + 0, s0);
    part_put(part, warp * 3 + 1, s1);
    part_put(part, warp * 3 + 2, s2);
  }
  g.sync();
  // lanes 0..2 of the group's first warp reduce one sum each over the group's warps
  const int w0 = g.first >> 5, nw = g.size >> 5;
  if (g.tid() < 3) {
    const int which = g.tid();
    __int128 v = 0;
    for (int w = w0; w < w0 + nw; ++w)
      v += (__int128)(((unsigned __int128)part.hi[w * 3 + which] << 64) | part.lo[w * 3 + which]);
    if (mode == 0) {
      if (which == 0) int128_to_big(v, b0, rec->l1);
      if (which == 1) int128_to_big(v, b1, rec->s2);
      if (which == 0) rec->flags_l = 0u;
    } else {
      if (which == 0) int128_to_big(v, b0, rec->a);
      if (which == 1) int128_to_big(v, b1, rec->b);
      if (which == 2) int128_to_big(v, b2, rec->p);
      if (which == 0) rec->flags_s = 0u;
    }
  }
  g.sync();
  return true;
}

// Exact sums of one row by a group: the 128-bit windows when the row's fp32
// sums are trustworthy and its terms fit, else the group's first warp runs
// the digit accumulator (non-finite or extreme rows).
__device__ __forceinline__ void exact_row_any(const SelectArgs &a, long long row, int mode, const float *st,
                                              ExactRec *rec, Part128 &part, const Group &g) {
  const bool trusted = mode == 0 ? !isnan(key_r(st)) : !isnan(key_s(st));
  bool ok = false;
  if (trusted)
    ok = a.dtype == TR_BF16  ? exact_row_block<TR_BF16>(a, row, mode, st, rec, part, g)
         : a.dtype == TR_F16 ? exact_row_block<TR_F16>(a, row, mode, st, rec, part, g)
                             : exact_row_block<TR_F32>(a, row, mode, st, rec, part, g);
  if (!ok) {
    if (g.tid() < 32) exact_row(a, row, mode, rec, threadIdx.x & 31);
    g.sync();
  }
}

// ---------------------------------------------------------------- double-float tier
// A near-tie is almost never an exact tie: the fp32 keys' bound (about
// 2^-22) is what leaves it open.  Before recomputing a row exactly, the
// select kernel recomputes its sums with error-free transformations -- every
// term, exact in fp32 (|x|, and squares and products of bf16 / fp16 values;
// fp32 squares and products as TwoProd pairs), enters a double-float by
// TwoSum -- and keeps the keys R and s as double-floats within Bounds::df_*
// (about 2^-32 relative or tighter).  A run whose rows these keys separate
// pairwise is ranked by them; one they do not separate (an exact tie, or
// closer than the bound) is recomputed exactly.  A row whose values could
// make a term inexact (a non-finite value, a square or product that would
// leave the normal fp32 range) or whose sums leave [kTiny, kHuge] is not
// handled here: it goes to the exact path.

// Runs longer than this skip the tier: long runs are exact ties in practice.
constexpr int kDfRunMax = 32;

// Value of element i of a 16-byte chunk as fp32 (exact for all three types).
template <int kDt>
__device__ __forceinline__ void unpack_f32(const uint4 &v, float *out) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if (kDt == TR_BF16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i] = __uint_as_float(w[i] << 16);
      out[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  } else if (kDt == TR_F16) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t h = (w[i >> 1] >> (16 * (i & 1))) & 0xffffu;
      const uint32_t sg = (h & 0x8000u) << 16, ex = (h >> 10) & 0x1fu, mant = h & 0x3ffu;
      float f;
      if (ex == 0x1fu)
        f = __uint_as_float(sg | 0x7f800000u | (mant << 13));
      else if (ex == 0u)
        f = __uint_as_float(sg | __float_as_uint(__uint2float_rn(mant) * 0x1p-24f));
      else
        f = __uint_as_float(sg | ((ex + 112u) << 23) | (mant << 13));
      out[i] = f;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) out[i] = __uint_as_float(w[i]);
  }
}

// A value whose square (and whose products with other such values) is an
// exact normal fp32 number or zero: 0, or 2^-50 <= |v| <= 2^50.
__device__ __forceinline__ bool df_value_ok(float v) {
  const float m = fabsf(v);
  return m == 0.f || (m >= 0x1p-50f && m <= 0x1p+50f);
}

// hi + lo += t with hi + (exact errors) the exact running sum.
__device__ __forceinline__ void df_term(float &hi, float &lo, float t) {
  const df::F2 r = df::two_sum(hi, t);
  hi = r.h;
  lo = __fadd_rn(lo, r.l);
}
__device__ __forceinline__ void df_join(float &hi, float &lo, float h2, float l2) {
  const df::F2 r = df::two_sum(hi, h2);
  hi = r.h;
  lo = __fadd_rn(__fadd_rn(lo, l2), r.l);
}
__device__ __forceinline__ void df_warp_join(float &hi, float &lo) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float h2 = __shfl_xor_sync(0xffffffffu, hi, o), l2 = __shfl_xor_sync(0xffffffffu, lo, o);
    df_join(hi, lo, h2, l2);
  }
}

struct PartDf {
  float h[kWarps * 3], l[kWarps * 3];
  int ok[4];  // per group: the row's keys were written
};

// Double-float keys of one row (mode 0: R from L1, S2 of x; mode 1: s from
// A, B, P of x', x'') by a group of warps; writes rec->r_* or rec->s_* and
// returns true, uniformly across the group, or false when the row is not
// eligible (nothing written).
template <int kDt>
__device__ __noinline__ bool df_row_block(const SelectArgs &a, long long row, int mode, ExactRec *rec, PartDf &part,
                                          const Group g) {
  constexpr int kPer = kDt == TR_F32 ? 4 : 8;  // elements per 16-byte chunk
  constexpr int kLoads = 2;                    // chunks per stream in flight per thread
  const int nchunks = a.d / kPer;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  bool ok = true;
  float h0 = 0.f, l0 = 0.f, h1 = 0.f, l1 = 0.f, h2 = 0.f, l2 = 0.f;
  const uint4 *p0 = static_cast<const uint4 *>(mode == 0 ? a.x : (a.x_pre ? a.x_pre : a.x)) + row * nchunks;
  const uint4 *p1 = static_cast<const uint4 *>(a.x_post) + row * nchunks;
  for (int c0 = g.tid(); c0 < nchunks; c0 += kLoads * g.size) {
    uint4 u0[kLoads], u1[kLoads];
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {  // every load of the round first
      const int c = c0 + j * g.size;
      if (c < nchunks) {
        u0[j] = __ldg(p0 + c);
        if (mode != 0) u1[j] = __ldg(p1 + c);
      }
    }
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      if (c0 + j * g.size >= nchunks) break;
      float v0[kPer], v1[kPer];
      unpack_f32<kDt>(u0[j], v0);
      if (mode == 0) {
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
          const float x = v0[i];
          ok &= df_value_ok(x);
          df_term(h0, l0, fabsf(x));
          if (kDt == TR_F32) {
            const df::F2 q = df::two_prod(x, x);
            df_term(h1, l1, q.h);
            l1 = __fadd_rn(l1, q.l);
          } else {
            df_term(h1, l1, __fmul_rn(x, x));
          }
        }
      } else {
        unpack_f32<kDt>(u1[j], v1);
#pragma unroll
        for (int i = 0; i < kPer; ++i) {
          const float p = v0[i], q = v1[i];
          ok &= df_value_ok(p) && df_value_ok(q);
          if (kDt == TR_F32) {
            const df::F2 pp2 = df::two_prod(p, p), qq2 = df::two_prod(q, q), pq2 = df::two_prod(p, q);
            df_term(h0, l0, pp2.h);
            l0 = __fadd_rn(l0, pp2.l);
            df_term(h1, l1, qq2.h);
            l1 = __fadd_rn(l1, qq2.l);
            df_term(h2, l2, pq2.h);
            l2 = __fadd_rn(l2, pq2.l);
          } else {
            df_term(h0, l0, __fmul_rn(p, p));
            df_term(h1, l1, __fmul_rn(q, q));
            df_term(h2, l2, __fmul_rn(p, q));
          }
        }
      }
    }
  }
  if (!g.all(ok)) return false;
  df_warp_join(h0, l0);
  df_warp_join(h1, l1);
  if (mode != 0) df_warp_join(h2, l2);
  if (lane == 0) {
    part.h[warp * 3 + 0] = h0;
    part.l[warp * 3 + 0] = l0;
    part.h[warp * 3 + 1] = h1;
    part.l[warp * 3 + 1] = l1;
    part.h[warp * 3 + 2] = h2;
    part.l[warp * 3 + 2] = l2;
  }
  g.sync();
  const int gi = g.bar - 1;
  const int w0 = g.first >> 5, nw = g.size >> 5;
  if (g.tid() < (mode == 0 ? 2 : 3)) {
    // thread j of the group's first warp merges sum j's warp partials in
    // turn, into the first warp's slot (only thread j touches index j)
    const int j = g.tid();
    float h = part.h[w0 * 3 + j], l = part.l[w0 * 3 + j];
    for (int w = w0 + 1; w < w0 + nw; ++w) df_join(h, l, part.h[w * 3 + j], part.l[w * 3 + j]);
    const df::F2 n = df::two_sum(h, l);
    part.h[w0 * 3 + j] = n.h;
    part.l[w0 * 3 + j] = n.l;
  }
  if (g.tid() < 32) __syncwarp();
  if (g.tid() == 0) {
    float s[3][2];
#pragma unroll
    for (int j = 0; j < 3; ++j) {
      s[j][0] = part.h[w0 * 3 + j];
      s[j][1] = part.l[w0 * 3 + j];
    }
    bool fine;
    if (mode == 0) {
      const df::F2 L1{s[0][0], s[0][1]}, S2{s[1][0], s[1][1]};
      fine = S2.h >= kTiny && S2.h <= kHuge;
      if (fine) {
        const df::F2 r = df::div(df::mul(L1, L1), S2);
        rec->r_hi = r.h;
        rec->r_lo = r.l;
      }
    } else {
      const df::F2 A{s[0][0], s[0][1]}, B{s[1][0], s[1][1]}, P{s[2][0], s[2][1]};
      fine = A.h >= kTiny && A.h <= kHuge && B.h >= kTiny && B.h <= kHuge;
      if (fine) {
        const df::F2 v = df::div(P, df::mul(df::sqrt(A), df::sqrt(B)));
        rec->s_hi = v.h;
        rec->s_lo = v.l;
      }
    }
    part.ok[gi] = fine ? 1 : 0;
  }
  g.sync();
  return part.ok[gi] != 0;
}

// +1 / -1 when the double-float keys order row a above / below row b for
// certain, 0 when their bounds overlap.
__device__ __forceinline__ int df_cmp_r(const ExactRec &ra, const ExactRec &rb, const Bounds &bd) {
  const float ah = ra.r_hi, bh = rb.r_hi;
  const float d = __fadd_rn(__fsub_rn(ah, bh), __fsub_rn(ra.r_lo, rb.r_lo));
  const float m = bd.df_r * (fabsf(ah) + fabsf(bh));
  return d > m ? 1 : (d < -m ? -1 : 0);
}
__device__ __forceinline__ int df_cmp_s(const ExactRec &ra, const ExactRec &rb, const Bounds &bd) {
  const float ah = ra.s_hi, bh = rb.s_hi;
  const float d = __fadd_rn(__fsub_rn(ah, bh), __fsub_rn(ra.s_lo, rb.s_lo));
  const float m = 2.f * bd.df_s_abs + bd.df_s_rel * (fabsf(ah) + fabsf(bh));
  return d > m ? 1 : (d < -m ? -1 : 0);
}

__device__ __forceinline__ bool df_row_any(const SelectArgs &a, long long row, int mode, ExactRec *rec, PartDf &part,
                                           const Group &g) {
  return a.dtype == TR_BF16  ? df_row_block<TR_BF16>(a, row, mode, rec, part, g)
         : a.dtype == TR_F16 ? df_row_block<TR_F16>(a, row, mode, rec, part, g)
                             : df_row_block<TR_F32>(a, row, mode, rec, part, g);
}

// Recomputes the rows whose flags request it: by the double-float tier where
// F_DF allows it and the row qualifies (F_DF stays set), else exactly (F_XL,
// F_XS).  The pending rows are listed first (a block-wide vote skips everything when
// none is); then up to four rows at a time are handled by groups of warps.
constexpr int kPendCap = 512;
// Recomputes the rows list[0..cnt) (local indices, cnt <= kPendCap) as
// their flags request, up to four rows at a time by groups of warps.
// Called by the whole block; ends with a block barrier.
__device__ __noinline__ void refine_list(const SelectArgs &a, long long off, const int *list, const int cnt,
                                         uint8_t *fl, ExactRec *rec, const bool primary) {
  __shared__ Part128 part;
  __shared__ PartDf pdf;
  const int groups = cnt >= 4 ? 4 : (cnt >= 2 ? 2 : 1);
  const int gsize = (int)blockDim.x / groups;
  const int gi = (int)threadIdx.x / gsize;
  const Group g{gi * gsize, gsize, 1 + gi};
  for (int base = 0; base < cnt; base += groups) {
    if (base + gi < cnt) {
      const int row = list[base + gi];
      const uint8_t fr = fl[row];
      const float *st = a.stats + (off + row) * TR_STATS_WORDS;
      bool dl = false, ds = false;  // settled by the double-float tier
      if (fr & F_NEEDL) {
        if (fr & F_DF) dl = df_row_any(a, off + row, 0, rec + row, pdf, g);
        if (!dl) exact_row_any(a, off + row, 0, st, rec + row, part, g);
      }
      if (fr & F_NEEDS) {
        if (fr & F_DF) ds = df_row_any(a, off + row, 1, rec + row, pdf, g);
        if (!ds) exact_row_any(a, off + row, 1, st, rec + row, part, g);
      }
      if (g.tid() == 0 && (fr & (F_NEEDL | F_NEEDS))) {  // a listed row may request nothing
        uint8_t f = (uint8_t)(fr & ~(F_NEEDL | F_NEEDS | F_DF));
        if (fr & F_NEEDL) f |= dl ? F_DF : F_XL;
        if (fr & F_NEEDS) f |= ds ? F_DF : F_XS;
        fl[row] = f;
        const bool exact = ((fr & F_NEEDL) && !dl) || ((fr & F_NEEDS) && !ds);
        if (exact && a.status && primary) atomicAdd(&a.status[2], 1);
      }
    }
    __syncthreads();
  }
}

// Every row of the image whose flags request it, listed from the flags.
__device__ __noinline__ void refine_listed(const SelectArgs &a, long long off, int n, uint8_t *fl, ExactRec *rec,
                                           const bool primary) {
  __shared__ int plist[kPendCap];
  __shared__ int pcount;
  for (;;) {
    if (threadIdx.x == 0) pcount = 0;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      if (fl[i] & (F_NEEDL | F_NEEDS)) {
        const int slot = atomicAdd(&pcount, 1);
        if (slot < kPendCap) plist[slot] = i;
      }
    }
    __syncthreads();
    const int total = pcount;
    if (total == 0) break;
    refine_list(a, off, plist, min(total, kPendCap), fl, rec, primary);
    if (total <= kPendCap) break;  // otherwise list the rows still pending
  }
}
// The common case -- nothing pending -- costs one pass over the flags and a
// block vote; the work itself stays out of line.
__device__ __forceinline__ void refine_pending(const SelectArgs &a, long long off, int n, uint8_t *fl,
                                               ExactRec *rec, const bool primary) {
  bool any = false;
  for (int i = threadIdx.x; i < n; i += blockDim.x) any |= (fl[i] & (F_NEEDL | F_NEEDS)) != 0;
  if (__syncthreads_or(any)) refine_listed(a, off, n, fl, rec, primary);
}

// ---------------------------------------------------------------- exact comparisons
constexpr int kWide = 4 * kBigLimbs;
struct Wide {
  uint32_t l[kWide];
  int n;
  int e;
};
__device__ __forceinline__ void wide_from(const Big &b, Wide &w) {
  w.n = b.n;
  w.e = b.e;
  for (int i = 0; i < b.n; ++i) w.l[i] = b.l[i];
}
__device__ __forceinline__ void wide_one(Wide &w) {
  w.n = 1;
  w.e = 0;
  w.l[0] = 1u;
}
// out = a * b (magnitudes); a.n + b.n <= kWide at every call site.
__device__ void wide_mul(const Wide &a, const Wide &b, Wide &out) {
  if (a.n == 0 || b.n == 0) {
    out.n = 0;
    out.e = 0;
    return;
  }
  out.n = a.n + b.n;
  out.e = a.e + b.e;
  for (int i = 0; i < out.n; ++i) out.l[i] = 0u;
  for (int i = 0; i < a.n; ++i) {
    unsigned long long carry = 0;
    for (int j = 0; j < b.n; ++j) {
      const unsigned long long t = (unsigned long long)a.l[i] * b.l[j] + out.l[i + j] + carry;
      out.l[i + j] = (uint32_t)t;
      carry = t >> 32;
    }
    out.l[i + b.n] = (uint32_t)carry;
  }
  while (out.n > 0 && out.l[out.n - 1] == 0u) --out.n;
}
__device__ int wide_cmp(const Wide &x, const Wide &y) {
  if (x.n == 0 || y.n == 0) return (x.n != 0) - (y.n != 0);
  const int tx = 32 * (x.e + x.n) - __clz(x.l[x.n - 1]);
  const int ty = 32 * (y.e + y.n) - __clz(y.l[y.n - 1]);
  if (tx != ty) return tx > ty ? 1 : -1;
  const int hi = max(x.e + x.n, y.e + y.n) - 1, lo = min(x.e, y.e);
  for (int p = hi; p >= lo; --p) {
    const uint32_t u = (p >= x.e && p < x.e + x.n) ? x.l[p - x.e] : 0u;
    const uint32_t v = (p >= y.e && p < y.e + y.n) ? y.l[p - y.e] : 0u;
    if (u != v) return u > v ? 1 : -1;
  }
  return 0;
}

// sign(R_a - R_b), R = L1^2 / S2 (R = 1 for an all-zero row, non-finite rows
// lowest), by big-integer cross products.
__device__ __noinline__ int cmp_r_big(const ExactRec &ra, const ExactRec &rb) {
  const bool na = ra.flags_l & kRecNonFiniteX, nb = rb.flags_l & kRecNonFiniteX;
  if (na || nb) return na == nb ? 0 : (na ? -1 : 1);
  Wide l1a, s2a, l1b, s2b, t, x, y;
  if (ra.l1.n == 0) {
    wide_one(l1a);
    wide_one(s2a);
  } else {
    wide_from(ra.l1, l1a);
    wide_from(ra.s2, s2a);
  }
  if (rb.l1.n == 0) {
    wide_one(l1b);
    wide_one(s2b);
  } else {
    wide_from(rb.l1, l1b);
    wide_from(rb.s2, s2b);
  }
  wide_mul(l1a, l1a, t);
  wide_mul(t, s2b, x);
  wide_mul(l1b, l1b, t);
  wide_mul(t, s2a, y);
  return wide_cmp(x, y);
}

// sign(s_a - s_b) through sigma = sign(P) P^2 / (A B) (s = 0 when A or B is 0,
// non-finite rows highest), by big-integer cross products.
__device__ __noinline__ int cmp_s_big(const ExactRec &ra, const ExactRec &rb) {
  const bool na = ra.flags_s & kRecNonFiniteS, nb = rb.flags_s & kRecNonFiniteS;
  if (na || nb) return na == nb ? 0 : (na ? 1 : -1);
  const int sa = (ra.a.n == 0 || ra.b.n == 0 || ra.p.n == 0) ? 0 : (ra.p.neg ? -1 : 1);
  const int sb = (rb.a.n == 0 || rb.b.n == 0 || rb.p.n == 0) ? 0 : (rb.p.neg ? -1 : 1);
  if (sa != sb) return sa > sb ? 1 : -1;
  if (sa == 0) return 0;
  Wide pa, aa, ba, pb, ab, bb, t, u, x, y;
  wide_from(ra.p, pa);
  wide_from(ra.a, aa);
  wide_from(ra.b, ba);
  wide_from(rb.p, pb);
  wide_from(rb.a, ab);
  wide_from(rb.b, bb);
  wide_mul(pa, pa, t);
  wide_mul(t, ab, u);
  wide_mul(u, bb, x);
  wide_mul(pb, pb, t);
  wide_mul(t, aa, u);
  wide_mul(u, ba, y);
  const int c = wide_cmp(x, y);
  return sa > 0 ? c : -c;
}

// The same comparisons screened first with 64-bit truncated mantissas
// (integer arithmetic only); only gaps below 2^-57 relative -- in practice
// exact ties -- go on to the big-integer cross products.
__device__ int cmp_r(const ExactRec &ra, const ExactRec &rb) {
  const bool na = ra.flags_l & kRecNonFiniteX, nb = rb.flags_l & kRecNonFiniteX;
  if (na || nb) return na == nb ? 0 : (na ? -1 : 1);
  const Fx l1a = ra.l1.n ? big_fx(ra.l1) : fx_one(), s2a = ra.l1.n ? big_fx(ra.s2) : fx_one();
  const Fx l1b = rb.l1.n ? big_fx(rb.l1) : fx_one(), s2b = rb.l1.n ? big_fx(rb.s2) : fx_one();
  const int c = fx_cmp(fx_mul(fx_mul(l1a, l1a), s2b), fx_mul(fx_mul(l1b, l1b), s2a));
  return c ? c : cmp_r_big(ra, rb);
}
__device__ int cmp_s(const ExactRec &ra, const ExactRec &rb) {
  const bool na = ra.flags_s & kRecNonFiniteS, nb = rb.flags_s & kRecNonFiniteS;
  if (na || nb) return na == nb ? 0 : (na ? 1 : -1);
  const int sa = (ra.a.n == 0 || ra.b.n == 0 || ra.p.n == 0) ? 0 : (ra.p.neg ? -1 : 1);
  const int sb = (rb.a.n == 0 || rb.b.n == 0 || rb.p.n == 0) ? 0 : (rb.p.neg ? -1 : 1);
  if (sa != sb) return sa > sb ? 1 : -1;
  if (sa == 0) return 0;
  const Fx pa = big_fx(ra.p), pb = big_fx(rb.p);
  const Fx x = fx_mul(fx_mul(fx_mul(pa, pa), big_fx(rb.a)), big_fx(rb.b));
  const Fx y = fx_mul(fx_mul(fx_mul(pb, pb), big_fx(ra.a)), big_fx(ra.b));
  const int c = fx_cmp(x, y);
  return c ? c * sa : cmp_s_big(ra, rb);
}

// ---------------------------------------------------------------- block helpers

__device__ int block_exclusive_scan(int v, int *total) {
  __shared__ int wsum[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  __syncthreads();  // wsum may still be read by a previous call
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nwarps ? wsum[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    wsum[lane] = w;
  }
  __syncthreads();
  *total = wsum[nwarps - 1];
  return (warp ? wsum[warp - 1] : 0) + x - v;
}

// Stable ascending LSD radix sort (8-bit digits) of the m rows listed in a
// by key[row]; b is scratch of the same size and hist holds kWarps x 256
// counters.  Warp w owns the contiguous stretch w of the current order:
// per-warp digit counts, a column scan (digit-major, then warp), then each
// warp scatters its stretch in order, ranking equal digits within 32 lanes
// with match-any, which keeps the sort stable.  A pass whose digit is the
// same for every row is skipped.  Returns the buffer holding the order.
__device__ __noinline__ uint16_t *radix_sort(const uint32_t *key, uint16_t *a, uint16_t *b, int m, uint32_t *hist) {
  __shared__ int skip;
  __shared__ uint32_t dsum[8];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int seg = (m + kWarps - 1) / kWarps;
  const int s0 = min(m, warp * seg), s1 = min(m, s0 + seg);
  uint32_t *h = hist + warp * 256;
  const unsigned lt = (1u << lane) - 1u;
  if (m < 2) return a;
#pragma unroll 1
  for (int shift = 0; shift < 32; shift += 8) {
    for (int d = lane; d < 256; d += 32) h[d] = 0u;
    if (tid == 0) skip = 0;
    __syncwarp();
    for (int q = s0 + lane; q < s1; q += 32) atomicAdd(&h[(key[a[q]] >> shift) & 0xffu], 1u);
    __syncthreads();
    uint32_t total = 0;
    if (tid < 256) {
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t c = hist[w * 256 + tid];
        hist[w * 256 + tid] = total;
        total += c;
      }
      if (total == (uint32_t)m) skip = 1;
    }
    uint32_t incl = total;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (tid < 256 && lane == 31) dsum[warp] = incl;
    __syncthreads();
    if (tid < 256) {
      uint32_t base = 0;
      for (int w = 0; w < warp; ++w) base += dsum[w];
      const uint32_t excl = base + incl - total;
      for (int w = 0; w < kWarps; ++w) hist[w * 256 + tid] += excl;
    }
    __syncthreads();
    if (!skip) {
      for (int q0 = s0; q0 < s1; q0 += 32) {
        const int q = q0 + lane;
        const bool act = q < s1;
        const unsigned am = __ballot_sync(0xffffffffu, act);
        if (act) {
          const uint16_t row = a[q];
          const uint32_t d = (key[row] >> shift) & 0xffu;
          const unsigned peers = __match_any_sync(am, d);
          const int rank = __popc(peers & lt);
          const uint32_t base = h[d];
          b[base + rank] = row;
          __syncwarp(am);
          if (rank == 0) h[d] = base + __popc(peers);
        }
        __syncwarp();
      }
      uint16_t *t = a;
      a = b;
      b = t;
    }
    __syncthreads();
  }
  return a;
}

// Ascending bitonic sort of kSelectThreads * E composite keys (sort key << 16
// | row) held E per thread (thread t owns positions t E .. t E + E - 1).
// For each merge size k the stages run with partner distance j = k/2, k/4,
// ..., 1: distances of at least 32 E go through shared memory (scratch:
// kSelectThreads * E words) between block barriers, distances of at least E
// through register shuffles inside a warp, and the last ones (j < E) inside
// the thread, with compile-time j so that v[] stays in registers.
template <int E>
__device__ void bitonic_regs(unsigned long long (&v)[E], unsigned long long *scratch) {
  constexpr int NP = kSelectThreads * E;
  const int t = threadIdx.x, lane = t & 31;
  for (int k = 2; k <= NP; k <<= 1) {
    for (int j = k >> 1; j >= E; j >>= 1) {
      if (j < 32 * E) {
        const int lm = j / E;
        const bool lower = (lane & lm) == 0;
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const unsigned long long o = __shfl_xor_sync(0xffffffffu, v[e], lm);
          const bool up = ((t * E + e) & k) == 0;
          v[e] = (lower == up) ? min(v[e], o) : max(v[e], o);
        }
      } else {
#pragma unroll
        for (int e = 0; e < E; ++e) scratch[t * E + e] = v[e];
        __syncthreads();
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int i = t * E + e, pi = i ^ j;
          const unsigned long long o = scratch[pi];
          const bool up = (i & k) == 0;
          v[e] = ((i < pi) == up) ? min(v[e], o) : max(v[e], o);
        }
        __syncthreads();
      }
    }
#pragma unroll
    for (int j = E >> 1; j > 0; j >>= 1) {
      if (j < k) {
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int pe = e ^ j;
          if (pe > e) {
            const bool up = ((t * E + e) & k) == 0;
            const unsigned long long x = v[e], y = v[pe];
            if ((x > y) == up) {
              v[e] = y;
              v[pe] = x;
            }
          }
        }
      }
    }
  }
}

// Ascending order of the m <= kSelectThreads rows listed in a by their
// composite keys (distinct), by counting: thread i places row a[i] at the
// number of listed rows with a smaller key.  m^2 comparisons spread over m
// threads and two block barriers: cheaper than a bitonic network for the
// short lists it takes (see kCountSortMax).  scratch: m 64-bit words,
// 16-byte aligned.
constexpr int kCountSortMax = 128;
__device__ void sort_count(const uint32_t *key, uint16_t *a, int m, unsigned long long *scratch) {
  const int tid = threadIdx.x;
  unsigned long long c = 0;
  if (tid < m) {
    c = ((unsigned long long)key[a[tid]] << 16) | a[tid];
    scratch[tid] = c;
  }
  if (tid == m && (m & 1)) scratch[m] = ~0ull;  // pads the last pair; never below c
  __syncthreads();
  if (tid < m) {
    const ulonglong2 *s2 = reinterpret_cast<const ulonglong2 *>(scratch);
    int rank = 0;
#pragma unroll 4
    for (int j = 0; j < (m + 1) >> 1; ++j) {
      const ulonglong2 v = s2[j];
      rank += (v.x < c) + (v.y < c);
    }
    a[rank] = (uint16_t)(c & 0xffffu);  // every read of a[] preceded the barrier
  }
  __syncthreads();
}

template <int E>
__device__ void sort_small(const uint32_t *key, uint16_t *a, int m, unsigned long long *scratch) {
  unsigned long long v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = threadIdx.x * E + e;
    v[e] = i < m ? (((unsigned long long)key[a[i]] << 16) | a[i]) : ~0ull;
  }
  __syncthreads();  // every thread has read its rows of a before they are overwritten
  bitonic_regs<E>(v, scratch);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = threadIdx.x * E + e;
    if (i < m) a[i] = (uint16_t)(v[e] & 0xffffu);
  }
  __syncthreads();
}

// ---------------------------------------------------------------- sorting
// Every sort orders rows by the composite (key[row] << 16 | row): by key, ties
// to the lower row (rows fit 16 bits), which is the order a stable sort of a
// row-ascending list gives.
__device__ __forceinline__ unsigned long long comp_key(const uint32_t *key, uint16_t row) {
  return ((unsigned long long)key[row] << 16) | row;
}

// The 511 splitters are kept in breadth-first (Eytzinger) order: node e has
// children 2e+1 and 2e+2, and an in-order walk visits them ascending.  The
// nodes a search can reach at one level are contiguous, so the lanes of a
// warp hit distinct banks (a sorted array searched by halving would send
// them all to the same few banks at the middle levels).
// In-order rank r (0..510) of the node at breadth-first index e:
// level l = floor(log2(e + 1)), place p = e + 1 - 2^l, r = (2p + 1) 2^(8 - l) - 1;
// inversely, with z the trailing zeros of r + 1: l = 8 - z, p = (r + 1) >> (z + 1).
__device__ __forceinline__ int eytzinger_index(int r) {
  const int z = __ffs(r + 1) - 1;
  return (1 << (8 - z)) - 1 + ((r + 1) >> (z + 1));
}
// Number of splitters below c: nine comparisons down the tree; the leaf
// reached, counted from the left, is that number.
__device__ __forceinline__ int splitter_rank(const unsigned long long *sp, unsigned long long c) {
  int e = 0;
#pragma unroll
  for (int l = 0; l < 9; ++l) e = 2 * e + 1 + (sp[e] < c ? 1 : 0);
  return e - 511;
}

// Sample sort of the m rows listed in a (1024 < m <= 16384) by composite key.
// kSelectThreads rows, one at a pseudo-random place inside each of
// kSelectThreads equal stretches of a (stratified: evenly spread, yet not
// aliased with periodic structure such as frames of equal length), are
// sorted (bitonic); all but the smallest split the keys into kSelectThreads
// buckets of about m / kSelectThreads rows each.  Each row finds its bucket
// once (kept in bid), rows are counted per bucket, the counts scanned, the
// rows scattered into their buckets (any order inside), and a row's place
// inside its bucket is the number of bucket members with a smaller composite
// key.  Returns the buffer holding the order, or nullptr, having changed
// nothing, when the buckets are so uneven that the in-bucket counting would
// cost more than kSampleWork comparisons per row on average, or hold more
// than kSampleBucketMax rows in one bucket (the caller then falls back to
// the radix sort).
// hist: kWarps x 256 words (splitters and bucket counters); bid: m entries.
constexpr int kSampleWork = 256;
constexpr int kSampleBucketMax = 512;
__device__ __forceinline__ uint32_t mix32(uint32_t x) {  // an integer hash (xorshift-multiply finaliser)
  x ^= x >> 16;
  x *= 0x7feb352du;
  x ^= x >> 15;
  x *= 0x846ca68bu;
  x ^= x >> 16;
  return x;
}
__device__ __noinline__ uint16_t *sample_sort(const uint32_t *key, uint16_t *a, uint16_t *b, uint16_t *bid, int m,
                                 uint32_t *hist) {
  static_assert(kSelectThreads == 512, "511 splitters, 512 buckets");
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  unsigned long long *sp = reinterpret_cast<unsigned long long *>(hist);  // [511] splitters (after the sample sort)
  uint32_t *cnt = hist + 2 * kSelectThreads;                             // [512] bucket counters
  unsigned long long v[1];
  {
    const int lo = (int)((long long)tid * m / kSelectThreads), hi = (int)((long long)(tid + 1) * m / kSelectThreads);
    v[0] = comp_key(key, a[lo + (int)(mix32((uint32_t)tid + 0x9e3779b9u) % (uint32_t)(hi - lo))]);
  }
  __syncthreads();  // hist may still be read by the caller's previous step
  bitonic_regs<1>(v, sp);
  if (tid) sp[eytzinger_index(tid - 1)] = v[0];
  cnt[tid] = 0u;
  __syncthreads();
  for (int q = tid; q < m; q += nthr) {
    const int k = splitter_rank(sp, comp_key(key, a[q]));
    bid[q] = (uint16_t)k;
    atomicAdd(&cnt[k], 1u);
  }
  __syncthreads();
  const int size = (int)cnt[tid];
  if (__syncthreads_or(size > kSampleBucketMax)) return nullptr;
  int total = 0;
  const int start = block_exclusive_scan(size, &total);
  int work = 0;  // sum of squared bucket sizes, at most m^2 <= 2^28
  block_exclusive_scan(size * size, &work);
  if ((long long)work > (long long)kSampleWork * m) return nullptr;  // uniform: work is block-wide
  cnt[tid] = (uint32_t)start;
  __syncthreads();
  for (int q = tid; q < m; q += nthr) b[atomicAdd(&cnt[bid[q]], 1u)] = a[q];
  __syncthreads();
  // cnt[k] is now the end of bucket k, which spans [cnt[k - 1], cnt[k]).
  // Warp w owns buckets 32w .. 32w + 31, contiguous in b; lane j holds the
  // end of bucket 32w + j, and each lane takes one position of the warp's
  // stretch per round: its bucket by a five-step shuffle search over the
  // ends, its place by counting the bucket's members with a smaller key.
  static_assert(kSelectThreads == 32 * kWarps, "one bucket per lane");
  const int end_l = (int)cnt[warp * 32 + lane];
  const int beg_w = warp ? (int)cnt[warp * 32 - 1] : 0;
  const int end_w = __shfl_sync(0xffffffffu, end_l, 31);
  for (int i0 = beg_w; i0 < end_w; i0 += 32) {
    const int i = min(i0 + lane, end_w - 1);
    int k = 0;  // number of this warp's buckets ending at or before i (at most 31)
#pragma unroll
    for (int step = 16; step >= 1; step >>= 1)
      if (__shfl_sync(0xffffffffu, end_l, k + step - 1) <= i) k += step;
    const int lo_s = __shfl_sync(0xffffffffu, end_l, max(k - 1, 0));
    const int lo = k ? lo_s : beg_w, hi = __shfl_sync(0xffffffffu, end_l, k);
    if (i0 + lane < end_w) {
      const uint16_t row = b[i];
      const unsigned long long c = comp_key(key, row);
      int rank = 0, q = lo;
      for (; q + 4 <= hi; q += 4) {  // four independent loads per step
        const uint16_t r0 = b[q], r1 = b[q + 1], r2 = b[q + 2], r3 = b[q + 3];
        rank += (comp_key(key, r0) < c ? 1 : 0) + (comp_key(key, r1) < c ? 1 : 0) +
                (comp_key(key, r2) < c ? 1 : 0) + (comp_key(key, r3) < c ? 1 : 0);
      }
      for (; q < hi; ++q) rank += comp_key(key, b[q]) < c ? 1 : 0;
      a[lo + rank] = row;
    }
  }
  __syncthreads();
  return a;
}

// Ascending order of the m rows listed in a by (key[row], row), by value
// buckets: the float each key encodes (v = value, or -value for importance
// keys, which are stored complemented) is mapped linearly from [vmin, vmax]
// onto nb buckets -- a monotone map, so concatenated buckets are in order --
// rows are scattered into their bucket (in b) with shared-memory atomics,
// and each row's final place is its bucket's start plus the number of
// bucket members with a smaller (key, row), counted by one thread per row
// (buckets hold about one row on the workloads here, at most kBucketMax).
// Returns a, holding the order, or nullptr, having changed nothing, when
// some bucket would hold more than kBucketMax rows (ties, or keys crowded
// together), a key encodes NaN, or the keys span no usable range: the caller
// then takes another sort.  hist: at least nb words.
constexpr int kBucketMax = 32;
constexpr int kBuckets = 4096;
__device__ __forceinline__ float key_value(uint32_t k, bool complemented) {
  return complemented ? -unord32(~k) : unord32(k);
}
__device__ uint16_t *bucket_sort(const uint32_t *key, uint16_t *a, uint16_t *b, int m, uint32_t *hist,
                                 bool complemented) {
  __shared__ float sh_min[kWarps], sh_max[kWarps];
  __shared__ int sh_big;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float vmin = INFINITY, vmax = -INFINITY;
  bool nan = false;
  for (int q = tid; q < m; q += blockDim.x) {
    const float v = key_value(key[a[q]], complemented);
    vmin = fminf(vmin, v);
    vmax = fmaxf(vmax, v);
    nan |= v != v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, o));
    vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
  }
  if (lane == 0) {
    sh_min[warp] = vmin;
    sh_max[warp] = vmax;
  }
  int nb = 64;
  while (nb < m && nb < kBuckets) nb <<= 1;
  for (int c = tid; c < nb; c += blockDim.x) hist[c] = 0u;
  if (tid == 0) sh_big = 0;
  __syncthreads();
  if (__syncthreads_or(nan)) return nullptr;  // uniform; NaN has no place in a linear bucket map
  vmin = sh_min[0];
  vmax = sh_max[0];
  for (int w = 1; w < kWarps; ++w) {
    vmin = fminf(vmin, sh_min[w]);
    vmax = fmaxf(vmax, sh_max[w]);
  }
  const float span = vmax - vmin;
  const float scale = (float)nb / span;
  if (!(span > 0.f) || !isfinite(span) || !isfinite(scale)) return nullptr;  // uniform: all equal or no usable range
  // bucket of a value: floor((v - vmin) * scale), monotone in v, clamped to the last bucket
  auto bucket = [&](float v) { return min(nb - 1, (int)((v - vmin) * scale)); };
  for (int q = tid; q < m; q += blockDim.x) atomicAdd(&hist[bucket(key_value(key[a[q]], complemented))], 1u);
  __syncthreads();
  // exclusive scan of the bucket counts (each thread a contiguous stretch) and the largest count
  const int per = (nb + blockDim.x - 1) / blockDim.x;
  const int c0 = min(nb, tid * per), c1 = min(nb, c0 + per);
  int run = 0, big = 0;
  for (int c = c0; c < c1; ++c) {
    run += (int)hist[c];
    big = max(big, (int)hist[c]);
  }
  if (big > kBucketMax) sh_big = 1;
  int total = 0;
  int base = block_exclusive_scan(run, &total);
  if (sh_big) return nullptr;  // uniform: written before the scan's barriers
  for (int c = c0; c < c1; ++c) {
    const int cnt = (int)hist[c];
    hist[c] = (uint32_t)base;
    base += cnt;
  }
  __syncthreads();
  for (int q = tid; q < m; q += blockDim.x) {
    const uint16_t row = a[q];
    b[atomicAdd(&hist[bucket(key_value(key[row], complemented))], 1u)] = row;
  }
  __syncthreads();
  // hist[c] is now the end of bucket c, so bucket c spans [hist[c - 1], hist[c])
  for (int q = tid; q < m; q += blockDim.x) {
    const uint16_t row = b[q];
    const uint32_t kr = key[row];
    const int c = bucket(key_value(kr, complemented));
    const int lo = c ? (int)hist[c - 1] : 0, hi = (int)hist[c];
    const unsigned long long kk = ((unsigned long long)kr << 16) | row;
    int rank = 0;
    for (int j = lo; j < hi; ++j) {
      const uint16_t r2 = b[j];
      rank += (((unsigned long long)key[r2] << 16) | r2) < kk;
    }
    a[lo + rank] = row;
  }
  __syncthreads();
  return a;
}

// Ascending order of the m rows listed in a by (key[row], row), a listed in
// ascending row order: a register bitonic sort up to 512 rows; above that
// value buckets, and when the values crowd into few buckets a register
// bitonic sort up to 2048 rows, the sample sort above, and the stable radix
// sort when the sample sort declines too.  Returns the buffer holding the
// order.
__device__ uint16_t *sort_rows(const uint32_t *key, uint16_t *a, uint16_t *b, uint16_t *bid, int m,
                               uint32_t *hist, bool complemented) {
  if (m < 2) return a;
  unsigned long long *scratch = reinterpret_cast<unsigned long long *>(hist);
  if (m <= kSelectThreads) {
    __syncthreads();  // hist may still be read by the caller's previous step
    if (m <= kCountSortMax)
      sort_count(key, a, m, scratch);
    else
      sort_small<1>(key, a, m, scratch);
    return a;
  }
  if (uint16_t *o = bucket_sort(key, a, b, m, hist, complemented)) return o;
  if (m <= 2 * kSelectThreads) {
    __syncthreads();
    sort_small<2>(key, a, m, scratch);
    return a;
  }
  if (m <= 4 * kSelectThreads) {
    __syncthreads();
    sort_small<4>(key, a, m, scratch);
    return a;
  }
  if (uint16_t *o = sample_sort(key, a, b, bid, m, hist)) return o;
  return radix_sort(key, a, b, m, hist);
}

// ---------------------------------------------------------------- selection
// Relative half-width of the window of importance values around an uncertain
// top-K1 cut whose rows are ordered first (about 2000 times the
// certification band of the keys).
constexpr float kCutWindow = 0x1p-11f;

// Key at position r (0-based) of the ascending order of key[0..n), found
// without sorting: four rounds of 8-bit digit histograms, most significant
// digit first, each over the rows whose higher digits equal those found so
// far.  *lt receives how many keys are smaller, *eq how many are equal.
// hist: kWarps x 256 words.  Called by the whole block.
__device__ uint32_t select_rank(const uint32_t *key, int n, int r, uint32_t *hist, int *lt, int *eq) {
  __shared__ uint32_t sh_pre;
  __shared__ int sh_r, sh_eq;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t pre = 0u, mask = 0u;
  int rr = r;
  __syncthreads();  // hist may still be read by the caller's previous step
#pragma unroll 1
  for (int shift = 24; shift >= 0; shift -= 8) {
    uint32_t *h = hist + warp * 256;
    for (int d = lane; d < 256; d += 32) h[d] = 0u;
    __syncwarp();
    for (int i = tid; i < n; i += blockDim.x) {
      const uint32_t k = key[i];
      if ((k & mask) == pre) atomicAdd(&h[(k >> shift) & 0xffu], 1u);
    }
    __syncthreads();
    if (tid < 256) {  // column tid: only this thread reads or writes it here
      uint32_t c = 0u;
      for (int w = 0; w < kWarps; ++w) c += hist[w * 256 + tid];
      hist[tid] = c;
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t c[8], sum = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c[j] = hist[lane * 8 + j];
        sum += c[j];
      }
      uint32_t incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      uint32_t acc = incl - sum;
      if (acc <= (uint32_t)rr && (uint32_t)rr < incl) {  // exactly one lane holds rank rr
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if ((uint32_t)rr < acc + c[j]) {
            sh_pre = pre | ((uint32_t)(lane * 8 + j) << shift);
            sh_r = rr - (int)acc;
            sh_eq = (int)c[j];
            break;
          }
          acc += c[j];
        }
      }
    }
    __syncthreads();
    pre = sh_pre;
    rr = sh_r;
    mask |= 0xffu << shift;
  }
  *lt = r - rr;
  *eq = sh_eq;
  return pre;
}

// The same selection by value buckets, in one pass over the keys instead of
// four: the value each key encodes (-R for the complemented importance
// keys, so ascending keys are ascending values) is mapped linearly from
// [vmin, vmax] onto nb buckets (a monotone map: equal keys share a bucket,
// and a smaller key never lands in a later bucket); a scan of the bucket
// counts finds the bucket holding position r, and one warp ranks its
// members.  Returns false, having set nothing, when the values span no
// usable range or that bucket holds more than 32 keys (the caller then
// takes the radix selection).  hist: at least kBuckets words.
__device__ bool select_rank_buckets(const uint32_t *key, int n, int r, uint32_t *hist, float vmin, float vmax,
                                    uint32_t *t_out, int *lt, int *eq) {
  __shared__ int sh_c, sh_before, sh_cnt, sh_lt, sh_eq;
  __shared__ uint32_t sh_mem[32], sh_t;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31;
  int nb = 64;
  while (nb < n && nb < kBuckets) nb <<= 1;
  const float span = vmax - vmin, scale = (float)nb / span;
  if (!(span > 0.f) || !isfinite(span) || !isfinite(scale)) return false;  // uniform
  auto bucket = [&](uint32_t k) { return min(nb - 1, max(0, (int)((key_value(k, true) - vmin) * scale))); };
  __syncthreads();  // hist may still be read by the caller's previous step
  for (int c = tid; c < nb; c += nthr) hist[c] = 0u;
  if (tid == 0) sh_cnt = 0;
  __syncthreads();
  for (int i = tid; i < n; i += nthr) atomicAdd(&hist[bucket(key[i])], 1u);
  __syncthreads();
  // the bucket holding position r: each thread sums a stretch of buckets
  const int per = (nb + nthr - 1) / nthr;
  const int c0 = min(nb, tid * per), c1 = min(nb, c0 + per);
  int run = 0;
  for (int c = c0; c < c1; ++c) run += (int)hist[c];
  int total = 0;
  int base = block_exclusive_scan(run, &total);
  if (base <= r && r < base + run) {
    for (int c = c0; c < c1; ++c) {
      const int h = (int)hist[c];
      if (r < base + h) {
        sh_c = c;
        sh_before = base;
        break;
      }
      base += h;
    }
  }
  __syncthreads();
  const int cstar = sh_c, before = sh_before, members = (int)hist[cstar];
  if (members > 32) return false;  // uniform
  for (int i = tid; i < n; i += nthr) {
    const uint32_t k = key[i];
    if (bucket(k) == cstar) sh_mem[atomicAdd(&sh_cnt, 1)] = k;
  }
  __syncthreads();
  if (tid < 32) {
    const uint32_t mk = lane < members ? sh_mem[lane] : 0xffffffffu;
    int less = 0, same = 0;
    for (int j = 0; j < members; ++j) {
      const uint32_t o = __shfl_sync(0xffffffffu, mk, j);
      less += o < mk;
      same += o == mk;
    }
    const int rr = r - before;  // position r inside the bucket
    if (lane < members && less <= rr && rr < less + same) {  // lanes holding equal keys write the same
      sh_t = mk;
      sh_lt = before + less;
      sh_eq = same;
    }
  }
  __syncthreads();
  *t_out = sh_t;
  *lt = sh_lt;
  *eq = sh_eq;
  return true;
}

// Block-wide minimum and maximum (every thread receives both).
__device__ void block_min_max(float &vmin, float &vmax) {
  __shared__ float smin[32], smax[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, o));
    vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, o));
  }
  __syncthreads();  // smin / smax may still be read by a previous call
  if (lane == 0) {
    smin[warp] = vmin;
    smax[warp] = vmax;
  }
  __syncthreads();
  vmin = smin[0];
  vmax = smax[0];
  for (int w = 1; w < nwarps; ++w) {
    vmin = fminf(vmin, smin[w]);
    vmax = fmaxf(vmax, smax[w]);
  }
}

// Smallest key[i] (i < n) above t, or 0xffffffff when there is none.
__device__ uint32_t block_min_above(const uint32_t *key, int n, uint32_t t) {
  __shared__ uint32_t wmin[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  uint32_t v = 0xffffffffu;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    const uint32_t k = key[i];
    if (k > t) v = min(v, k);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();  // wmin may still be read by a previous call
  if (lane == 0) wmin[warp] = v;
  __syncthreads();
  v = 0xffffffffu;
  for (int w = 0; w < nwarps; ++w) v = min(v, wmin[w]);
  return v;
}

__host__ __device__ inline int row_capacity(int max_n) { return (max_n + 15) / 16 * 16; }

// ---------------------------------------------------------------- one image
// Algorithm 1 for image b, by the whole CTA (kSelectThreads threads);
// Sorted position of diversity pick j < K2 among the M rows of X_rem:
// Algorithm 1's integer stride j t, or the real interval M / K2 of
// Section IV-B, floor(j M / K2).
__device__ __forceinline__ int pick_position(int j, int m, int k2, int t, bool interval) {
  return interval ? (int)((long long)j * m / k2) : j * t;
}
// Whether sorted position q of X_rem is one of the K2 picks.  For the
// interval the first pick at or after q is j = ceil(q K2 / M).
__device__ __forceinline__ bool is_pick(int q, int m, int k2, int t, bool interval) {
  if (!interval) return q % t == 0 && q / t < k2;
  const long long j = ((long long)q * k2 + m - 1) / m;
  return j < k2 && (j * m) / k2 == q;
}

// smem holds select_smem_bytes(a.max_n) bytes.  Reads the statistics through
// L2 so that rows scored by other CTAs of the same launch are seen.  Leaves
// the K kept local indices, ascending, in the second order buffer of smem
// (kept_rows); only a primary CTA writes idx, role, H2/s and the status words
// (replicas that run the same deterministic selection write nothing).
// The state of one image's selection in a CTA: where its rows are, its
// budgets and the CTA's shared-memory arrays (layout in select_smem_bytes).
// The uncertain runs of one image's decisions, kept so that their rows are
// recomputed and ranked without passes over every row: a run is a stretch
// [lo, hi) of sorted positions, packed (lo << 16) | hi.
constexpr int kMaxRuns = 128;
struct RunList {
  uint32_t run[kMaxRuns];
  int count, rows, longest;  // runs recorded (may exceed kMaxRuns), their rows, the longest
  int npend, npend2;         // rows listed for the first and second recomputation
  int list[kPendCap];
};

struct ImageCtx {
  long long off;
  int n, k, k1, k2, ko;
  bool need_r, need_s, primary;
  bool any_exact;    // some row was settled exactly up front
  float vmin, vmax;  // range of -R32 over the rows with a float key
  uint32_t *key, *hist;
  uint16_t *ia, *ib, *bid;
  uint8_t *fl;
  const float *st;
  ExactRec *rec;
  RunList *runs;  // block-shared
};

// Sets up c for image b; false when there is nothing to select (an invalid
// budget, counted in status[3] by the primary CTA, or an empty image).
__device__ __forceinline__ bool image_ctx(const SelectArgs &a, const int b, unsigned char *smem, const bool primary,
                                          ImageCtx &c) {
  const int tid = threadIdx.x;
  long long off;
  int n;
  if (a.cu_seqlens) {
    off = a.cu_seqlens[b];
    n = a.cu_seqlens[b + 1] - a.cu_seqlens[b];
  } else {
    off = (long long)b * a.n_uniform;
    n = a.n_uniform;
  }
  const int k = a.k[b], k1 = a.k1[b];
  // an image whose rows lie outside the packed tensors (malformed
  // cu_seqlens) is skipped like an invalid budget: nothing is read or written
  if (n < 0 || n > a.max_n || off < 0 || off + n > a.total_rows || k < 0 || k > n || k1 < 0 || k1 > k) {
    if (tid == 0 && a.status && primary) atomicAdd(&a.status[3], 1);
    return false;
  }
  if (n == 0) return false;
  const int cap = row_capacity(a.max_n);
  c.off = off;
  c.n = n;
  c.k = k;
  c.k1 = k1;
  c.k2 = k - k1;
  c.ko = a.cu_k[b];
  c.need_r = k1 > 0 && k1 < n;  // the importance order decides something
  c.need_s = k - k1 > 0;
  c.primary = primary;
  c.key = reinterpret_cast<uint32_t *>(smem);                          // [cap] sort key per row
  c.ia = reinterpret_cast<uint16_t *>(c.key + cap);                    // [cap] order buffers
  c.ib = c.ia + cap;                                                   // [cap]
  c.hist = reinterpret_cast<uint32_t *>(c.ib + cap);                   // [kWarps x 256]
  c.bid = reinterpret_cast<uint16_t *>(c.hist + kWarps * 256);         // [cap] sort scratch
  c.fl = reinterpret_cast<uint8_t *>(c.bid + cap);                     // [cap] row flags
  c.st = a.stats + off * TR_STATS_WORDS;
  c.rec = a.exact + off;
  return true;
}

// 1. Rows whose fp32 sums left the error model are settled exactly first
//    (also when only their H2 / s outputs need it): the importance side
//    (want_l) and / or the consistency side (want_s).  The same pass lays
//    out the importance keys ~ord32(R32) and the identity order.
__device__ __forceinline__ void settle_unreliable(const SelectArgs &a, ImageCtx &c, const bool want_l,
                                                  const bool want_s) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  const long long off = c.off;
  uint32_t *key = c.key;
  uint16_t *ia = c.ia;
  uint8_t *fl = c.fl;
  const float *st = c.st;
  ExactRec *rec = c.rec;
  const bool primary = c.primary;
  const bool need_r = c.need_r, need_s = c.need_s;
  bool any = false;
  float vmin = INFINITY, vmax = -INFINITY;
  for (int i0 = tid; i0 < n; i0 += kKeyIlp * nthr) {
    float2 kk[kKeyIlp];
#pragma unroll
    for (int u = 0; u < kKeyIlp; ++u) {
      const int i = i0 + u * nthr;
      kk[u] = i < n ? key_rs(st + (long long)i * TR_STATS_WORDS) : make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kKeyIlp; ++u) {
      const int i = i0 + u * nthr;
      if (i < n) {
        uint8_t f = 0;
        if (want_l && (need_r || a.h2) && isnan(kk[u].x)) f |= F_NEEDL;
        if (want_s && (need_s || a.s) && isnan(kk[u].y)) f |= F_NEEDS;
        any |= f != 0;
        fl[i] = f;
        key[i] = ~ord32(kk[u].x);
        ia[i] = (uint16_t)i;
        if (kk[u].x == kk[u].x) {  // the value stage I's bucket map sees: -R
          vmin = fminf(vmin, -kk[u].x);
          vmax = fmaxf(vmax, -kk[u].x);
        }
      }
    }
  }
  block_min_max(vmin, vmax);  // its barriers also publish fl, key and ia
  c.vmin = vmin;
  c.vmax = vmax;
  c.any_exact = __syncthreads_or(any);
  if (c.any_exact) {
    refine_listed(a, off, n, fl, rec, primary);
    __syncthreads();
  }
}

// Stage I when the K1-th and (K1+1)-th keys are not certainly ordered (t1:
// the K1-th key).  Out of line: only images with a near-tie at the cut come
// here.
__device__ __noinline__ void resolve_cut(const SelectArgs &a, const ImageCtx c, const uint32_t t1) {
  __shared__ int sh_lo, sh_hi;
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  const long long off = c.off;
  uint32_t *key = c.key;
  uint32_t *hist = c.hist;
  uint16_t *ia = c.ia;
  uint16_t *ib = c.ib;
  uint16_t *bid = c.bid;
  uint8_t *fl = c.fl;
  ExactRec *rec = c.rec;
  const bool primary = c.primary;
  const int k1 = c.k1;
  // Uncertain cut: only the order near it matters.  The rows whose R32
  // lies within a relative kCutWindow of the K1-th one (far wider than
  // the certification band) are listed and sorted; when the uncertain
  // run around the cut ends inside that list, every row with a smaller
  // key (larger R) precedes it in the full order and is certainly kept,
  // every row with a larger key certainly not.  Otherwise (or when the
  // window holds too many rows) all n rows are sorted.
  const float r1 = unord32(~t1);
  const uint32_t kw_lo = ~ord32(r1 * (1.f + kCutWindow)), kw_hi = ~ord32(r1 * (1.f - kCutWindow));
  const bool windowed = isfinite(r1) && r1 > 0.f;  // uniform
  const uint16_t *ord = nullptr;
  int base = 0, len = 0;  // ord[q] sits at position base + q of the full order
  if (windowed) {
    const int per = (n + nthr - 1) / nthr;
    const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
    int c_in = 0, c_lt = 0;
    for (int i = i0; i < i1; ++i) {
      const uint32_t k = key[i];
      c_in += k >= kw_lo && k <= kw_hi;
      c_lt += k < kw_lo;
      // above the window, R exceeds the K1-th key's by far more than the
      // keys' bound: certainly among the K1 kept, whichever order follows
      if (k < kw_lo) fl[i] |= F_IMP;
    }
    // one scan of both counts (each total is at most n < 2^16)
    int both = 0;
    int pos = block_exclusive_scan(c_in | (c_lt << 16), &both) & 0xffff;
    const int n_in = both & 0xffff, n_lt = both >> 16;
    if (n_in <= 2 * kSelectThreads) {  // uniform
      for (int i = i0; i < i1; ++i) {
        const uint32_t k = key[i];
        if (k >= kw_lo && k <= kw_hi) ib[pos++] = (uint16_t)i;
      }
      __syncthreads();
      unsigned long long *scratch = reinterpret_cast<unsigned long long *>(hist);
      if (n_in <= kCountSortMax)
        sort_count(key, ib, n_in, scratch);
      else if (n_in <= kSelectThreads)
        sort_small<1>(key, ib, n_in, scratch);
      else
        sort_small<2>(key, ib, n_in, scratch);
      ord = ib;
      base = n_lt;
      len = n_in;
    }
  }
  for (int attempt = 0; attempt < 2; ++attempt) {
    if (!ord) {
      ord = sort_rows(key, ia, ib, bid, n, hist, true);
      base = 0;
      len = n;
    }
    const bool whole = base == 0 && len == n;
    // The uncertain run around position p = k1 - base: from the last
    // certified boundary at or before p (0 if none) to the first at or after
    // p (len if none), found by all threads at once; a certified p gives
    // lo = hi = p, no run.
    const int p = k1 - base;
    const bool outside = p < 1 || p >= len;  // uniform
    if (tid == 0) {
      sh_lo = 0;
      sh_hi = len;
    }
    __syncthreads();
    if (!outside) {
      int my_lo = 0, my_hi = len;
      for (int q = 1 + tid; q < len; q += nthr)
        if (cert_r(key, ord, q, a.bounds)) {
          if (q <= p) my_lo = q;  // q rises: the last one wins
          if (q >= p && my_hi == len) my_hi = q;
        }
      if (my_lo > 0) atomicMax(&sh_lo, my_lo);
      if (my_hi < len) atomicMin(&sh_hi, my_hi);
    }
    __syncthreads();
    if (tid == 0) {
      if (outside) {
        sh_lo = -1;
        sh_hi = p;
      } else if (sh_lo != sh_hi && !whole && (sh_lo == 0 || sh_hi == len)) {
        sh_lo = -1;  // the run may go on outside the list
      }
    }
    __syncthreads();
    if (sh_lo >= 0) break;
    ord = nullptr;  // the window was not enough: sort everything
  }
  const int lo = sh_lo, hi = sh_hi;
  for (int q = tid; q < lo; q += nthr) fl[ord[q]] |= F_IMP;
  if (hi > lo) {
    // The run's rows: double-float keys first (short runs), and exact
    // sums when those do not separate every pair or a row has them already.
    const uint8_t want = hi - lo <= kDfRunMax ? (uint8_t)(F_NEEDL | F_DF) : (uint8_t)F_NEEDL;
    for (int q = lo + tid; q < hi; q += nthr) {
      const int r = ord[q];
      if (!(fl[r] & F_XL)) fl[r] |= want;
      if (hi - lo <= kPendCap) c.runs->list[q - lo] = r;  // rows with nothing requested are left alone
    }
    __syncthreads();
    if (hi - lo <= kPendCap)
      refine_list(a, off, c.runs->list, hi - lo, fl, rec, primary);
    else
      refine_pending(a, off, n, fl, rec, primary);
    __syncthreads();
    bool open = false;
    for (int q = lo + tid; q < hi && !open; q += nthr) {
      const int r = ord[q];
      open = (fl[r] & F_XL) != 0;
      for (int q2 = q + 1; q2 < hi && !open; ++q2) {
        const int r2 = ord[q2];
        open = (fl[r2] & F_XL) || df_cmp_r(rec[r2], rec[r], a.bounds) == 0;
      }
    }
    if (__syncthreads_or(open)) {
      for (int q = lo + tid; q < hi; q += nthr) {
        const int r = ord[q];
        if (!(fl[r] & F_XL)) fl[r] = (uint8_t)((fl[r] & ~F_DF) | F_NEEDL);
      }
      __syncthreads();
      if (hi - lo <= kPendCap)
        refine_list(a, off, c.runs->list, hi - lo, fl, rec, primary);
      else
        refine_pending(a, off, n, fl, rec, primary);
      __syncthreads();
    }
    for (int q = lo + tid; q < hi; q += nthr) {
      const int r = ord[q];
      const bool exact = (fl[r] & F_XL) != 0;  // then every row of the run is
      const bool ovf = exact && (rec[r].flags_l & kRecOverflowL);
      int rank = 0;
      for (int q2 = lo; q2 < hi; ++q2) {
        if (q2 == q) continue;
        const int r2 = ord[q2];
        int c;
        if (!exact)
          c = df_cmp_r(rec[r2], rec[r], a.bounds);  // never 0 here
        else if (ovf || (rec[r2].flags_l & kRecOverflowL))
          c = q2 < q ? 1 : -1;  // no exact value: keep the float order
        else
          c = cmp_r(rec[r2], rec[r]);
        if (c > 0 || (c == 0 && r2 < r)) ++rank;
      }
      if (base + lo + rank < k1) fl[r] |= F_IMP;
    }
  }
  __syncthreads();
}

// 2. Stage I: top-K1 by R (equivalently H2), descending, lower index first.
//    Marks X_imp (F_IMP) in the flags.
__device__ __forceinline__ void stage_one(const SelectArgs &a, ImageCtx &c) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  uint32_t *key = c.key;
  uint32_t *hist = c.hist;
  uint8_t *fl = c.fl;
  ExactRec *rec = c.rec;
  const int k1 = c.k1;
  const bool need_r = c.need_r;
  if (need_r) {
    if (c.any_exact) {  // rows settled exactly carry their exact key (the
                        // bucket map clamps it into range: still monotone)
      for (int i = tid; i < n; i += nthr)
        if (fl[i] & F_XL) key[i] = ~ord32(exact_r_key(rec[i]));
      __syncthreads();
    }
    const float vmin = c.vmin, vmax = c.vmax;
    // Fast path: the K1-th and (K1+1)-th keys (by value buckets, else radix
    // selection); when they differ and their order is certain, the top K1
    // are exactly the rows with a key up to the K1-th, and no order is needed.
    int lt = 0, eq = 0;
    uint32_t t1 = 0u;
    if (!select_rank_buckets(key, n, k1 - 1, hist, vmin, vmax, &t1, &lt, &eq))
      t1 = select_rank(key, n, k1 - 1, hist, &lt, &eq);
    bool settled = false;
    if (lt + eq == k1) {
      const uint32_t t2 = block_min_above(key, n, t1);
      settled = cert_r_val(unord32(~t1), unord32(~t2), a.bounds);
    }
    if (settled) {
      for (int i = tid; i < n; i += nthr)
        if (key[i] <= t1) fl[i] |= F_IMP;
      __syncthreads();
    } else {
      resolve_cut(a, c, t1);
    }
  } else if (k1 == n) {
    for (int i = tid; i < n; i += nthr) fl[i] |= F_IMP;
    __syncthreads();
  }
}

// 3a. Consistency keys ord32(s32) of every row (stage I's keys are no
//     longer needed; X_imp rows' keys are never read), exact ones for
//     settled rows.
__device__ __forceinline__ void consistency_keys(const SelectArgs &a, ImageCtx &c) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  uint32_t *key = c.key;
  uint8_t *fl = c.fl;
  const float *st = c.st;
  ExactRec *rec = c.rec;
    for (int i0 = tid; i0 < n; i0 += kKeyIlp * nthr) {
    float sv[kKeyIlp];
#pragma unroll
    for (int u = 0; u < kKeyIlp; ++u) {
      const int i = i0 + u * nthr;
      sv[u] = i < n ? key_s(st + (long long)i * TR_STATS_WORDS) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < kKeyIlp; ++u) {
      const int i = i0 + u * nthr;
      if (i < n) {
        const uint8_t f = fl[i];
        key[i] = ord32((f & F_XS) ? exact_s_key(rec[i]) : sv[u]);
        fl[i] = (uint8_t)(f & ~F_DF);  // a stage-I double-float key is not an s key
      }
    }
  }
}

// The rows of the image (all, or those outside X_imp) in ascending index
// order -- the stable sort's tie order -- into dst; returns their number.
__device__ __forceinline__ int list_rows(ImageCtx &c, uint16_t *dst, const bool skip_imp) {
  const int tid = threadIdx.x, nthr = blockDim.x, n = c.n;
  const uint8_t *fl = c.fl;
  const int per = (n + nthr - 1) / nthr;
  const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += !(skip_imp && (fl[i] & F_IMP));
  int m = 0;
  int pos = block_exclusive_scan(cnt, &m);
  for (int i = i0; i < i1; ++i)
    if (!(skip_imp && (fl[i] & F_IMP))) dst[pos++] = (uint16_t)i;
  __syncthreads();
  return m;
}

// Stage II's uncertain neighbourhoods (rows flagged F_RUN): each run is
// ranked by double-float keys or, failing those, exactly, and the stride
// picks inside it are marked.  Out of line: only images with a near-tie at a
// pick come here.  This version passes over every sorted position; the one
// below works from the recorded runs and takes over when they are few and
// short.
__device__ __noinline__ void rank_pick_runs_all(const SelectArgs &a, const ImageCtx c, const uint16_t *ord,
                                                const int m, const int t) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  const long long off = c.off;
  uint32_t *key = c.key;
  uint8_t *fl = c.fl;
  ExactRec *rec = c.rec;
  const bool primary = c.primary;
  const int k2 = c.k2;
  refine_pending(a, off, n, fl, rec, primary);
  __syncthreads();
  // A run whose double-float keys leave a pair unseparated (or with a row
  // that has exact sums) is recomputed exactly as a whole.
  bool open = false;
  for (int q = tid; q < m; q += nthr) {
    const int r = ord[q];
    if (!(fl[r] & F_RUN) || (fl[r] & F_XS)) continue;
    int lo = q;
    while (lo > 0 && !cert_s(key, ord, lo, a.bounds)) --lo;
    int hi = q + 1;
    while (hi < m && !cert_s(key, ord, hi, a.bounds)) ++hi;
    bool undecided = false;
    for (int q2 = lo; q2 < hi && !undecided; ++q2) {
      if (q2 == q) continue;
      const int r2 = ord[q2];
      undecided = (fl[r2] & F_XS) || df_cmp_s(rec[r2], rec[r], a.bounds) == 0;
    }
    if (undecided) {
      open = true;
      for (int q2 = lo; q2 < hi; ++q2) {
        const int r2 = ord[q2];
        if (!(fl[r2] & F_XS)) fl[r2] = (uint8_t)((fl[r2] & ~F_DF) | F_NEEDS);
      }
    }
  }
  if (__syncthreads_or(open)) {
    refine_pending(a, off, n, fl, rec, primary);
    __syncthreads();
  }
  for (int q = tid; q < m; q += nthr) {
    const int r = ord[q];
    if (!(fl[r] & F_RUN)) continue;
    int lo = q;
    while (lo > 0 && !cert_s(key, ord, lo, a.bounds)) --lo;
    int hi = q + 1;
    while (hi < m && !cert_s(key, ord, hi, a.bounds)) ++hi;
    const bool exact = (fl[r] & F_XS) != 0;  // then every row of the run is
    const bool ovf = exact && (rec[r].flags_s & kRecOverflowS);
    int rank = 0;
    for (int q2 = lo; q2 < hi; ++q2) {
      if (q2 == q) continue;
      const int r2 = ord[q2];
      int c;
      if (!exact)
        c = df_cmp_s(rec[r2], rec[r], a.bounds);  // never 0 here
      else if (ovf || (rec[r2].flags_s & kRecOverflowS))
        c = q2 < q ? -1 : 1;
      else
        c = cmp_s(rec[r2], rec[r]);
      if (c < 0 || (c == 0 && r2 < r)) ++rank;
    }
    if (is_pick(lo + rank, m, k2, t, a.stride_interval)) fl[r] |= F_DIV;
  }
  __syncthreads();
}

// The recorded runs: their rows are listed directly (no pass over all
// positions), recomputed, checked pairwise and ranked, one thread per run.
__device__ __noinline__ void rank_pick_runs(const SelectArgs &a, const ImageCtx c, const uint16_t *ord, const int m,
                                            const int t) {
  RunList &rl = *c.runs;
  const int nruns = rl.count;
  if (nruns > kMaxRuns || rl.rows > kPendCap || rl.longest > kDfRunMax) {  // uniform
    rank_pick_runs_all(a, c, ord, m, t);
    return;
  }
  const int tid = threadIdx.x, nthr = blockDim.x;
  uint8_t *fl = c.fl;
  ExactRec *rec = c.rec;
  const int k2 = c.k2;
  // 1. the runs' rows that request a recomputation (double-float first)
  for (int r = tid; r < nruns; r += nthr) {
    const int lo = (int)(rl.run[r] >> 16), hi = (int)(rl.run[r] & 0xffffu);
    for (int q = lo; q < hi; ++q) {
      const int row = ord[q];
      if (fl[row] & F_NEEDS) rl.list[atomicAdd(&rl.npend, 1)] = row;
    }
  }
  __syncthreads();
  if (rl.npend) refine_list(a, c.off, rl.list, rl.npend, fl, rec, c.primary);
  // 2. a run whose double-float keys leave a pair unseparated (or with a
  //    row that has exact sums) is recomputed exactly as a whole
  for (int r = tid; r < nruns; r += nthr) {
    const int lo = (int)(rl.run[r] >> 16), hi = (int)(rl.run[r] & 0xffffu);
    bool undecided = false;
    for (int q = lo; q < hi && !undecided; ++q) {
      const int r1 = ord[q];
      undecided = (fl[r1] & F_XS) != 0;
      for (int q2 = q + 1; q2 < hi && !undecided; ++q2) {
        const int r2 = ord[q2];
        undecided = (fl[r2] & F_XS) || df_cmp_s(rec[r2], rec[r1], a.bounds) == 0;
      }
    }
    if (undecided) {
      for (int q = lo; q < hi; ++q) {
        const int row = ord[q];
        if (!(fl[row] & F_XS)) {
          fl[row] = (uint8_t)((fl[row] & ~F_DF) | F_NEEDS);
          rl.list[atomicAdd(&rl.npend2, 1)] = row;
        }
      }
    }
  }
  __syncthreads();
  if (rl.npend2) refine_list(a, c.off, rl.list, rl.npend2, fl, rec, c.primary);
  // 3. ranks inside each run (every row of a run is double-float, or every
  //    row exact), and the picks among them
  for (int r = tid; r < nruns; r += nthr) {
    const int lo = (int)(rl.run[r] >> 16), hi = (int)(rl.run[r] & 0xffffu);
    for (int q = lo; q < hi; ++q) {
      const int row = ord[q];
      const bool exact = (fl[row] & F_XS) != 0;
      const bool ovf = exact && (rec[row].flags_s & kRecOverflowS);
      int rank = 0;
      for (int q2 = lo; q2 < hi; ++q2) {
        if (q2 == q) continue;
        const int r2 = ord[q2];
        int cmp;
        if (!exact)
          cmp = df_cmp_s(rec[r2], rec[row], a.bounds);  // never 0 here
        else if (ovf || (rec[r2].flags_s & kRecOverflowS))
          cmp = q2 < q ? -1 : 1;
        else
          cmp = cmp_s(rec[r2], rec[row]);
        if (cmp < 0 || (cmp == 0 && r2 < row)) ++rank;
      }
      if (is_pick(lo + rank, m, k2, t, a.stride_interval)) fl[row] |= F_DIV;
    }
  }
  __syncthreads();
}

// 3b. Stage II along ord, X_rem sorted by s (m rows): the stride picks
//     (F_DIV), with uncertain neighbourhoods settled exactly.
__device__ __forceinline__ void stage_two_picks(const SelectArgs &a, ImageCtx &c, const uint16_t *ord, const int m) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  uint32_t *key = c.key;
  uint8_t *fl = c.fl;
  const int k2 = c.k2;
  const int t = max(1, m / k2);
  bool marked = false;  // some pick's neighbourhood is uncertain
  for (int j = tid; j < k2; j += nthr) {
    const int p = pick_position(j, m, k2, t, a.stride_interval);
    const bool c0 = p == 0 || cert_s(key, ord, p, a.bounds);
    const bool c1 = p + 1 >= m || cert_s(key, ord, p + 1, a.bounds);
    if (c0 && c1) {
      fl[ord[p]] |= F_DIV;
    } else {
      int lo = p;
      while (lo > 0 && !cert_s(key, ord, lo, a.bounds)) --lo;
      int hi = p + 1;
      while (hi < m && !cert_s(key, ord, hi, a.bounds)) ++hi;
      // Threads whose runs coincide write the same bits: the races are benign.
      // Short runs try the double-float keys first.
      const uint8_t want = hi - lo <= kDfRunMax ? (uint8_t)(F_NEEDS | F_DF) : (uint8_t)F_NEEDS;
      for (int q = lo; q < hi; ++q) {
        const int r = ord[q];
        fl[r] |= (uint8_t)(F_RUN | ((fl[r] & F_XS) ? 0 : want));
      }
      marked = true;
      // every pick inside a run finds the same run; the first one records it
      if (j == 0 || pick_position(j - 1, m, k2, t, a.stride_interval) < lo) {
        RunList &rl = *c.runs;
        const int slot = atomicAdd(&rl.count, 1);
        if (slot < kMaxRuns) rl.run[slot] = ((uint32_t)lo << 16) | (uint32_t)hi;
        atomicAdd(&rl.rows, hi - lo);
        atomicMax(&rl.longest, hi - lo);
      }
    }
  }
  if (__syncthreads_or(marked)) rank_pick_runs(a, c, ord, m, t);  // else every pick is certain
}

// 4. X* = X_imp union X_div in ascending token order (Eq. 7), plus outputs;
//    the kept local indices are also left in ia (kept_rows).
__device__ __forceinline__ void emit_outputs(const SelectArgs &a, ImageCtx &c) {
  const int tid = threadIdx.x;
  const int nthr = blockDim.x;
  const int n = c.n;
  const long long off = c.off;
  uint16_t *ia = c.ia;
  uint8_t *fl = c.fl;
  ExactRec *rec = c.rec;
  const bool primary = c.primary;
  const int k = c.k, ko = c.ko;
  const int per = (n + nthr - 1) / nthr;
  const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += (fl[i] & (F_IMP | F_DIV)) != 0;
  int kept_total = 0;
  int pos = ko + block_exclusive_scan(cnt, &kept_total);
  for (int i = i0; i < i1; ++i) {
    const uint8_t f = fl[i];
    if ((f & (F_IMP | F_DIV)) && pos < ko + k) {  // never write past this image's slots
      if (primary) a.idx[pos] = i;
      ia[pos - ko] = (uint16_t)i;
      ++pos;
    }
    if (!primary) continue;
    if (a.role) a.role[off + i] = (f & F_IMP) ? 1 : ((f & F_DIV) ? 2 : 0);
    int nonfinite = 0, overflow = 0;
    if (f & F_XL) {
      const ExactRec &r = rec[i];
      nonfinite |= (r.flags_l & kRecNonFiniteX) != 0;
      overflow |= (r.flags_l & kRecOverflowL) != 0;
      if (a.h2 && !(r.flags_l & kRecOverflowL))
        a.h2[off + i] = exact_h2(r);
    }
    if (f & F_XS) {
      const ExactRec &r = rec[i];
      nonfinite |= (r.flags_s & kRecNonFiniteS) != 0;
      overflow |= (r.flags_s & kRecOverflowS) != 0;
      if (a.s && !(r.flags_s & kRecOverflowS))
        a.s[off + i] = (r.flags_s & kRecNonFiniteS) ? INFINITY : exact_s_key(r);
    }
    if (a.status) {
      if (nonfinite) atomicAdd(&a.status[0], 1);
      if (overflow) atomicAdd(&a.status[1], 1);
    }
  }
  if (tid == 0 && kept_total != k && a.status && primary) atomicAdd(&a.status[3], 1);
  __syncthreads();
}

// The selection of image b by one CTA (Algorithm 1 with exact decisions).
__device__ void select_image(const SelectArgs &a, const int b, unsigned char *smem, const bool primary = true) {
  __shared__ RunList runs;
  ImageCtx c;
  if (!image_ctx(a, b, smem, primary, c)) return;
  c.runs = &runs;
  settle_unreliable(a, c, true, true);
  stage_one(a, c);
  if (c.need_s) {
    if (threadIdx.x == 0) {  // read after the barriers of the listing and the sort
      runs.count = runs.rows = runs.longest = 0;
      runs.npend = runs.npend2 = 0;
    }
    consistency_keys(a, c);
    const int m = list_rows(c, c.ia, true);
    const uint16_t *ord = sort_rows(c.key, c.ia, c.ib, c.bid, m, c.hist, false);
    stage_two_picks(a, c, ord, m);
  }
  emit_outputs(a, c);
}

// Where select_image leaves the kept local indices.
__device__ __forceinline__ const uint16_t *kept_rows(const SelectArgs &a, unsigned char *smem) {
  return reinterpret_cast<const uint16_t *>(reinterpret_cast<uint32_t *>(smem) + row_capacity(a.max_n));
}

}  // namespace

size_t select_smem_bytes(int max_n);

}  // namespace tr
