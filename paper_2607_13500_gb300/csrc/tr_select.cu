// Selection of Algorithm 1 (Stage I top-K1 by H2, Stage II ascending sort by s
// and stride pick), one CTA per image, with exact decisions.
//
// Keys.  H2 = log R with R = L1^2 / S2 (Eq. 3-4: sum_j p_j^2 = S2 / L1^2),
// so ranking by H2 is ranking by R; s = P / sqrt(A B) (Eq. 6).  The CTA sorts
// fp32 keys R32 (descending) and s32 (ascending) built from the score pass's
// sums, packed with the token index into 64-bit words so that equal keys
// order by the lower index.
//
// Certification.  The score pass's sums carry proven error bounds (Bounds),
// so a cut between sorted neighbours is certain when their key intervals do
// not overlap; with a uniform relative (R) or monotone absolute (s) bound it
// suffices to test adjacent pairs.  Only decisions matter: the cut at K1 for
// Stage I and the neighbourhood of each stride position for Stage II.  The
// tokens of an uncertain run (a maximal stretch of uncertain cuts around a
// decision) are recomputed exactly -- their five sums as integers, from the
// input bits -- and ranked by exact rational comparison (cross products of
// big integers), ties to the lower index.  Rows whose fp32 sums left the
// error model (non-finite, overflowed, tiny) are recomputed exactly up front.
#include <cfloat>
#include <climits>
#include <cmath>

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
};

// ---------------------------------------------------------------- float keys
__device__ __forceinline__ uint32_t ord32(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unord32(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}
__device__ __forceinline__ int row_at(const unsigned long long *keys, int q) { return (int)(keys[q] & 0xffffffffu); }
__device__ __forceinline__ float r_at(const unsigned long long *keys, int q) {
  return unord32(~(uint32_t)(keys[q] >> 32));
}
__device__ __forceinline__ float s_at(const unsigned long long *keys, int q) {
  return unord32((uint32_t)(keys[q] >> 32));
}

__device__ __forceinline__ bool force_l(const float *st) {
  const float l1 = st[0], s2 = st[1];
  if (!(isfinite(l1) && isfinite(s2))) return true;
  return l1 != 0.f && (s2 < kTiny || s2 > kHuge);
}
__device__ __forceinline__ bool force_s(const float *st) {
  const float a = st[2], b = st[3], ph = st[4], pl = st[5];
  if (!(isfinite(a) && isfinite(b) && isfinite(ph) && isfinite(pl))) return true;
  return a < kTiny || b < kTiny || a > kHuge || b > kHuge;
}
__device__ __forceinline__ float approx_r(const float *st) {
  const float l1 = st[0], s2 = st[1];
  return l1 == 0.f ? 1.f : (float)((double)l1 * (double)l1 / (double)s2);
}
__device__ __forceinline__ float approx_s(const float *st) {
  return (float)(((double)st[4] + (double)st[5]) / sqrt((double)st[2] * (double)st[3]));
}

__device__ double big_to_double(const Big &b) {
  if (b.n == 0) return 0.0;
  const int top = b.n - 1, bot = b.n >= 3 ? b.n - 3 : 0;
  double v = 0.0;
  for (int i = top; i >= bot; --i) v = v * 4294967296.0 + (double)b.l[i];
  v = ldexp(v, 32 * (b.e + bot));
  return b.neg ? -v : v;
}
__device__ __forceinline__ double exact_r_value(const ExactRec &r) {
  if (r.flags_l & kRecNonFiniteX) return 0.0;
  if (r.l1.n == 0) return 1.0;
  const double l1 = big_to_double(r.l1);
  return l1 * l1 / big_to_double(r.s2);
}
__device__ __forceinline__ double exact_s_value(const ExactRec &r) {
  if (r.flags_s & kRecNonFiniteS) return 2.0;
  if (r.a.n == 0 || r.b.n == 0) return 0.0;
  return big_to_double(r.p) / sqrt(big_to_double(r.a) * big_to_double(r.b));
}

// Cut between importance-sorted positions q-1 and q (descending R32) is
// certain when R(q-1) > R(q) for every value the bounds allow.
__device__ __forceinline__ bool cert_r(const unsigned long long *keys, int q, double rho) {
  const double ra = r_at(keys, q - 1), rb = r_at(keys, q);
  return ra / (1.0 + rho) > rb / (1.0 - rho);
}
// Cut between consistency-sorted positions q-1 and q (ascending s32).
__device__ __forceinline__ bool cert_s(const unsigned long long *keys, int q, const Bounds &bd) {
  const double sa = s_at(keys, q - 1), sb = s_at(keys, q);
  const double ea = bd.es_abs + bd.es_rel * fabs(sa), eb = bd.es_abs + bd.es_rel * fabs(sb);
  return sa + ea < sb - eb;
}

// ---------------------------------------------------------------- exact sums
constexpr int kDig = 20;  // 32-bit digit positions per exact accumulator

struct Term {
  uint32_t m;  // integer significand
  int e;       // value = m * 2^e
  bool nonfinite;
};
__device__ __forceinline__ Term decode(const void *base, long long i, bool bf16) {
  Term t;
  if (bf16) {
    const uint32_t b = static_cast<const uint16_t *>(base)[i];
    const uint32_t ex = (b >> 7) & 0xffu, mant = b & 0x7fu;
    t.nonfinite = ex == 0xffu;
    t.m = ex ? (mant | 0x80u) : mant;
    t.e = (ex ? (int)ex : 1) - 134;
  } else {
    const uint32_t b = static_cast<const uint32_t *>(base)[i];
    const uint32_t ex = (b >> 23) & 0xffu, mant = b & 0x7fffffu;
    t.nonfinite = ex == 0xffu;
    t.m = ex ? (mant | 0x800000u) : mant;
    t.e = (ex ? (int)ex : 1) - 150;
  }
  return t;
}
__device__ __forceinline__ bool sign_bit(const void *base, long long i, bool bf16) {
  return bf16 ? (static_cast<const uint16_t *>(base)[i] >> 15) != 0 : (static_cast<const uint32_t *>(base)[i] >> 31) != 0;
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
  int hi = kDig + 1;
  while (hi >= 0 && limb[hi] == 0) --hi;
  out.neg = 0;
  if (hi < 0) {
    out.n = 0;
    out.e = 0;
    return true;
  }
  int lo = 0;
  while (limb[lo] == 0) ++lo;
  const int n = hi - lo + 1;
  if (n > kBigLimbs) {
    out.n = 0;
    out.e = 0;
    return false;
  }
  for (int i = 0; i < n; ++i) out.l[i] = limb[lo + i];
  out.n = (uint8_t)n;
  out.e = (int16_t)(lo + base / 32);
  out.neg = neg ? 1 : 0;
  return true;
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
// Digit bases (multiples of 32): |x| has exponent >= -133 (bf16) or -149
// (fp32), products >= -266 or -298; the top digit stays below kDig.
__device__ void exact_row(const SelectArgs &a, long long row, int mode, ExactRec *rec, int lane) {
  const bool bf16 = a.dtype == TR_BF16;
  const int base1 = -160;
  const int base2 = bf16 ? -288 : -320;
  long long d0[kDig], d1[kDig], d2[kDig];
  for (int k = 0; k < kDig; ++k) d0[k] = d1[k] = d2[k] = 0;
  bool nonfinite = false;
  const long long first = row * (long long)a.d;
  if (mode == 0) {
    for (int j = lane; j < a.d; j += 32) {
      const Term t = decode(a.x, first + j, bf16);
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
      const Term p = decode(xp, first + j, bf16);
      const Term q = decode(a.x_post, first + j, bf16);
      if (p.nonfinite || q.nonfinite) {
        nonfinite = true;
        continue;
      }
      if (p.m) add_term(d0, base2, (unsigned long long)p.m * p.m, 2 * p.e, false);
      if (q.m) add_term(d1, base2, (unsigned long long)q.m * q.m, 2 * q.e, false);
      if (p.m && q.m) {
        const bool neg = sign_bit(xp, first + j, bf16) != sign_bit(a.x_post, first + j, bf16);
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

// Every warp takes 32-row groups round-robin and recomputes the rows whose
// flags request it; clears the request and records what is now exact.
__device__ void refine_pending(const SelectArgs &a, long long off, int n, uint8_t *fl, ExactRec *rec) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  for (int g = warp; g * 32 < n; g += nwarps) {
    const int i = g * 32 + lane;
    const uint8_t f = i < n ? fl[i] : 0;
    unsigned mask = __ballot_sync(0xffffffffu, (f & (F_NEEDL | F_NEEDS)) != 0);
    while (mask) {
      const int r = __ffs(mask) - 1;
      mask &= mask - 1;
      const int row = g * 32 + r;
      const uint8_t fr = (uint8_t)__shfl_sync(0xffffffffu, (int)f, r);
      if (fr & F_NEEDL) exact_row(a, off + row, 0, rec + row, lane);
      if (fr & F_NEEDS) exact_row(a, off + row, 1, rec + row, lane);
      if (lane == 0) {
        fl[row] = (uint8_t)((fr & ~(F_NEEDL | F_NEEDS)) | ((fr & F_NEEDL) ? F_XL : 0) | ((fr & F_NEEDS) ? F_XS : 0));
        if (a.status) atomicAdd(&a.status[2], 1);
      }
    }
  }
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

// sign(R_a - R_b), R = L1^2 / S2 (R = 1 for an all-zero row, non-finite rows lowest).
__device__ int cmp_r(const ExactRec &ra, const ExactRec &rb) {
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
// non-finite rows highest).
__device__ int cmp_s(const ExactRec &ra, const ExactRec &rb) {
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

// ---------------------------------------------------------------- block helpers
__device__ void bitonic_sort(unsigned long long *keys, int np) {
  for (int k = 2; k <= np; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < np; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const unsigned long long u = keys[i], v = keys[ixj];
          const bool up = (i & k) == 0;
          if ((u > v) == up) {
            keys[i] = v;
            keys[ixj] = u;
          }
        }
      }
      __syncthreads();
    }
  }
}

__device__ int block_exclusive_scan(int v, int *total) {
  __shared__ int wsum[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
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

__host__ __device__ inline int next_pow2(int n) {
  int p = 1;
  while (p < n) p <<= 1;
  return p;
}

// ---------------------------------------------------------------- the kernel
__global__ void __launch_bounds__(kSelectThreads, 1) k_select(const SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int sh_lo, sh_hi;
  const int b = blockIdx.x;
  const int tid = threadIdx.x, nthr = blockDim.x;
  long long off;
  int n;
  if (a.cu_seqlens) {
    off = a.cu_seqlens[b];
    n = a.cu_seqlens[b + 1] - a.cu_seqlens[b];
  } else {
    off = (long long)b * a.n_uniform;
    n = a.n_uniform;
  }
  const int k = a.k[b], k1 = a.k1[b], k2 = k - k1, ko = a.cu_k[b];
  if (n < 0 || n > a.max_n || k < 0 || k > n || k1 < 0 || k1 > k) {
    if (tid == 0 && a.status) atomicAdd(&a.status[3], 1);
    return;
  }
  if (n == 0) return;
  const int np = next_pow2(n);
  unsigned long long *keys = reinterpret_cast<unsigned long long *>(smem);
  uint8_t *fl = reinterpret_cast<uint8_t *>(keys + next_pow2(a.max_n));
  const float *st = a.stats + off * TR_STATS_WORDS;
  ExactRec *rec = a.exact + off;
  const bool need_r = k1 > 0 && k1 < n;  // the importance order decides something
  const bool need_s = k2 > 0;

  // 1. Rows whose fp32 sums left the error model are settled exactly first
  //    (also when only their H2 / s outputs need it).
  for (int i = tid; i < n; i += nthr) {
    const float *r = st + (long long)i * TR_STATS_WORDS;
    uint8_t f = 0;
    if ((need_r || a.h2) && force_l(r)) f |= F_NEEDL;
    if ((need_s || a.s) && force_s(r)) f |= F_NEEDS;
    fl[i] = f;
  }
  __syncthreads();
  refine_pending(a, off, n, fl, rec);
  __syncthreads();

  // 2. Stage I: top-K1 by R (equivalently H2), descending, lower index first.
  if (need_r) {
    for (int i = tid; i < np; i += nthr) {
      unsigned long long key = ~0ull;
      if (i < n) {
        const float r = (fl[i] & F_XL) ? (float)exact_r_value(rec[i]) : approx_r(st + (long long)i * TR_STATS_WORDS);
        key = ((unsigned long long)(~ord32(r)) << 32) | (unsigned)i;
      }
      keys[i] = key;
    }
    __syncthreads();
    bitonic_sort(keys, np);
    if (tid == 0) {
      int lo = k1, hi = k1;
      if (!cert_r(keys, k1, a.bounds.rho_r)) {
        lo = k1 - 1;
        while (lo > 0 && !cert_r(keys, lo, a.bounds.rho_r)) --lo;
        hi = k1 + 1;
        while (hi < n && !cert_r(keys, hi, a.bounds.rho_r)) ++hi;
      }
      sh_lo = lo;
      sh_hi = hi;
    }
    __syncthreads();
    const int lo = sh_lo, hi = sh_hi;
    for (int q = tid; q < lo; q += nthr) fl[row_at(keys, q)] |= F_IMP;
    if (hi > lo) {
      for (int q = lo + tid; q < hi; q += nthr) {
        const int r = row_at(keys, q);
        if (!(fl[r] & F_XL)) fl[r] |= F_NEEDL;
      }
      __syncthreads();
      refine_pending(a, off, n, fl, rec);
      __syncthreads();
      for (int q = lo + tid; q < hi; q += nthr) {
        const int r = row_at(keys, q);
        const bool ovf = rec[r].flags_l & kRecOverflowL;
        int rank = 0;
        for (int q2 = lo; q2 < hi; ++q2) {
          if (q2 == q) continue;
          const int r2 = row_at(keys, q2);
          int c;
          if (ovf || (rec[r2].flags_l & kRecOverflowL))
            c = q2 < q ? 1 : -1;  // no exact value: keep the float order
          else
            c = cmp_r(rec[r2], rec[r]);
          if (c > 0 || (c == 0 && r2 < r)) ++rank;
        }
        if (lo + rank < k1) fl[r] |= F_IMP;
      }
    }
    __syncthreads();
  } else if (k1 == n) {
    for (int i = tid; i < n; i += nthr) fl[i] |= F_IMP;
    __syncthreads();
  }

  // 3. Stage II: sort X_rem by s ascending, pick positions 0, t, 2t, ...
  if (need_s) {
    const int m = n - k1;
    for (int i = tid; i < np; i += nthr) {
      unsigned long long key = ~0ull;
      if (i < n && !(fl[i] & F_IMP)) {
        const float sv = (fl[i] & F_XS) ? (float)exact_s_value(rec[i]) : approx_s(st + (long long)i * TR_STATS_WORDS);
        key = ((unsigned long long)ord32(sv) << 32) | (unsigned)i;
      }
      keys[i] = key;
    }
    __syncthreads();
    bitonic_sort(keys, np);
    const int t = max(1, m / k2);
    for (int j = tid; j < k2; j += nthr) {
      const int p = j * t;
      const bool c0 = p == 0 || cert_s(keys, p, a.bounds);
      const bool c1 = p + 1 >= m || cert_s(keys, p + 1, a.bounds);
      if (c0 && c1) {
        fl[row_at(keys, p)] |= F_DIV;
      } else {
        int lo = p;
        while (lo > 0 && !cert_s(keys, lo, a.bounds)) --lo;
        int hi = p + 1;
        while (hi < m && !cert_s(keys, hi, a.bounds)) ++hi;
        // Threads whose runs coincide write the same bits: the races are benign.
        for (int q = lo; q < hi; ++q) {
          const int r = row_at(keys, q);
          fl[r] |= (uint8_t)(F_RUN | ((fl[r] & F_XS) ? 0 : F_NEEDS));
        }
      }
    }
    __syncthreads();
    refine_pending(a, off, n, fl, rec);
    __syncthreads();
    for (int q = tid; q < m; q += nthr) {
      const int r = row_at(keys, q);
      if (!(fl[r] & F_RUN)) continue;
      int lo = q;
      while (lo > 0 && !cert_s(keys, lo, a.bounds)) --lo;
      int hi = q + 1;
      while (hi < m && !cert_s(keys, hi, a.bounds)) ++hi;
      const bool ovf = rec[r].flags_s & kRecOverflowS;
      int rank = 0;
      for (int q2 = lo; q2 < hi; ++q2) {
        if (q2 == q) continue;
        const int r2 = row_at(keys, q2);
        int c;
        if (ovf || (rec[r2].flags_s & kRecOverflowS))
          c = q2 < q ? -1 : 1;
        else
          c = cmp_s(rec[r2], rec[r]);
        if (c < 0 || (c == 0 && r2 < r)) ++rank;
      }
      const int pos = lo + rank;
      if (pos % t == 0 && pos / t < k2) fl[r] |= F_DIV;
    }
    __syncthreads();
  }

  // 4. X* = X_imp union X_div in ascending token order (Eq. 7), plus outputs.
  const int per = (n + nthr - 1) / nthr;
  const int i0 = min(n, tid * per), i1 = min(n, i0 + per);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += (fl[i] & (F_IMP | F_DIV)) != 0;
  int kept_total = 0;
  int pos = ko + block_exclusive_scan(cnt, &kept_total);
  for (int i = i0; i < i1; ++i) {
    const uint8_t f = fl[i];
    if ((f & (F_IMP | F_DIV)) && pos < ko + k) {  // never write past this image's slots
      a.idx[pos] = i;
      ++pos;
    }
    if (a.role) a.role[off + i] = (f & F_IMP) ? 1 : ((f & F_DIV) ? 2 : 0);
    int nonfinite = 0, overflow = 0;
    if (f & F_XL) {
      const ExactRec &r = rec[i];
      nonfinite |= (r.flags_l & kRecNonFiniteX) != 0;
      overflow |= (r.flags_l & kRecOverflowL) != 0;
      if (a.h2 && !(r.flags_l & kRecOverflowL))
        a.h2[off + i] = (r.flags_l & kRecNonFiniteX) ? -INFINITY : (float)log(exact_r_value(r));
    }
    if (f & F_XS) {
      const ExactRec &r = rec[i];
      nonfinite |= (r.flags_s & kRecNonFiniteS) != 0;
      overflow |= (r.flags_s & kRecOverflowS) != 0;
      if (a.s && !(r.flags_s & kRecOverflowS))
        a.s[off + i] = (r.flags_s & kRecNonFiniteS) ? INFINITY : (float)exact_s_value(r);
    }
    if (a.status) {
      if (nonfinite) atomicAdd(&a.status[0], 1);
      if (overflow) atomicAdd(&a.status[1], 1);
    }
  }
  if (tid == 0 && kept_total != k && a.status) atomicAdd(&a.status[3], 1);
}

int g_smem_set[64];  // per device: dynamic shared memory limit already raised

}  // namespace

size_t select_smem_bytes(int max_n) {
  return (size_t)next_pow2(max_n > 0 ? max_n : 1) * sizeof(unsigned long long) + align_up((size_t)max_n, 16);
}

cudaError_t launch_select(const SelectArgs &a, cudaStream_t st) {
  if (a.batch == 0) return cudaSuccess;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const size_t smem = select_smem_bytes(a.max_n);
  if (!g_smem_set[dev & 63]) {
    int optin = 0;
    err = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (err != cudaSuccess) return err;
    err = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - 1024);
    if (err != cudaSuccess) return err;
    g_smem_set[dev & 63] = 1;
  }
  k_select<<<a.batch, kSelectThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace tr
