// Internal declarations shared by the CUDA translation units of libtr.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <utility>

#include "tr.h"

namespace tr {

// ---------------------------------------------------------------- launch shapes
constexpr int kScoreWarps = 2;        // rows (one per warp) in flight per score CTA
constexpr int kScoreBatchBf16 = 8;    // 16-byte chunks a lane loads per stream before it computes (bf16)
constexpr int kScoreBatchF32 = 8;     // the same for fp32 inputs
constexpr int kSelectThreads = 512;   // one select CTA per image
constexpr int kGatherWarps = 8;

// ---------------------------------------------------------------- exact sums
// A non-negative integer magnitude times a power of two, with a sign:
//   value = (-1)^neg * sum_i l[i] * 2^(32 * (i + e)),  n limbs in use (n = 0 means 0).
constexpr int kBigLimbs = 8;
struct Big {
  uint32_t l[kBigLimbs];
  int16_t e;
  uint8_t n;
  uint8_t neg;
};

// Exact per-row sums of Eq. 3-4 (L1 = sum|x|, S2 = sum x^2) and of Eq. 6
// (P = sum x'x'', A = sum x'^2, B = sum x''^2).
enum : uint32_t {
  kRecNonFiniteX = 1u,   // x holds Inf/NaN: ranks last by importance
  kRecNonFiniteS = 2u,   // x' or x'' holds Inf/NaN: sorts last by s
  kRecOverflowL = 4u,    // L1 or S2 did not fit kBigLimbs limbs
  kRecOverflowS = 8u,    // P, A or B did not fit kBigLimbs limbs
};
struct ExactRec {
  Big l1, s2, a, b, p;
  uint32_t flags_l;  // kRecNonFiniteX | kRecOverflowL, valid once L1, S2 are filled
  uint32_t flags_s;  // kRecNonFiniteS | kRecOverflowS, valid once P, A, B are filled
  uint32_t pad;
  // The keys R and s recomputed in double-float from error-free sums
  // (hi + lo each; see the select kernel's double-float tier), within the
  // Bounds::df_* bounds of the true keys.
  float r_hi, r_lo, s_hi, s_lo;
};
static_assert(sizeof(ExactRec) % 16 == 0, "ExactRec records keep 16-byte alignment");

// ---------------------------------------------------------------- error bounds
// Rounding depth of the sums L1, S2, A, B in the score kernel: each term goes
// through the depth-3 (bf16) or depth-2 (fp32, plus the rounding of the square
// itself) tree of its 16-byte chunk; the chunk partials are accumulated
// error-free into double-floats (two per lane for bf16: even and odd chunks)
// whose low parts' own rounding is bounded separately (at most lane_chunks
// + 12 low-part additions on any path, folds and warp merges included), and
// the keys are computed from the unrounded double-float.
__host__ __device__ inline int elem_bytes(int dtype) { return dtype == TR_F32 ? 4 : 2; }

__host__ __device__ inline int score_depth(int d, int dtype) {
  (void)d;
  (void)dtype;
  return 3;
}

// Certification bounds for the float selection keys (see the select kernel):
//  * importance key R32 = fp32(L1^2 / S2): R32 = R (1 + delta), |delta| <= rho_r;
//  * consistency key s32 = fp32(P / sqrt(A B)): |s32 - s| <= es_abs + es_rel |s32|.
struct Bounds {
  double rho_r;
  double es_abs;
  double es_rel;
  // the same bounds as fp32 factors rounded outward, for tests evaluated
  // with directed rounding:  R >= R32 * r_lo,  R <= R32 * r_hi,
  // |s - s32| <= s_abs + s_rel |s32|
  float r_lo, r_hi, s_abs, s_rel;
  // Keys recomputed by the select kernel's double-float tier (R_df, s_df):
  // |R_df - R| <= df_r R_df,  |s_df - s| <= df_s_abs + df_s_rel |s_df|
  // (fp32, rounded outward).
  float df_r, df_s_abs, df_s_rel;
};

inline Bounds certification_bounds(int d, int dtype) {
  const double u = 1.0 / 16777216.0;  // fp32 unit roundoff 2^-24
  const int h = score_depth(d, dtype);
  const int per_chunk = 16 / elem_bytes(dtype);
  const double lane_chunks = (double)((d / per_chunk + 31) / 32);
  const double lane_terms = lane_chunks * per_chunk;
  // Double-float low parts: m additions of error terms each below u times the
  // running sum leave at most m^2 u^2 of the sum (m = the low part's additions).
  const double m = lane_chunks + 12.0;
  const double g = h * u / (1.0 - h * u) + m * m * u * u + 0x1p-34;  // relative error of L1, S2, A, B
  // P = P_hi + P_lo is exact up to the rounding of the P_lo additions:
  // at most u^2 (lane_terms^2 / 2 + 12 d) sum|x'x''| (doubled for fp32
  // inputs, whose product errors also enter P_lo; bf16 and fp16 products,
  // 16 and 22 significant bits, are exact), and sum|x'x''| <= sqrt(A B).
  double ep = 2.0 * u * u * (lane_terms * lane_terms + 12.0 * d) + 0x1p-52;
  if (dtype == TR_F32) ep *= 2.0;  // bf16 and fp16 products are exact in fp32
  // The encoder-MLP GEMM's epilogue (tr_mlp_score, bf16) writes the same
  // records: each term enters its double-float sum through TwoSum, over at
  // most 128 columns per partial (low-part roundings below
  // u^2 128 * 129 / 2 of the partial's sum|x'x''|), and the 2 ceil(d / 256)
  // partials are merged (2 roundings of at most u^2 129 of the total each);
  // the bound below, written for partials of up to 256 columns, covers that.
  // The bounds cover both producers of a record.  Its L1, S2, A and B are
  // within that same tiny relative error, far inside g below.
  if (dtype == TR_BF16) {
    const double col_blocks = (double)((d + 255) / 256);
    const double ep_mlp = u * u * (256.0 * 257.0 / 2.0 + 2.0 * 257.0 * col_blocks) + 0x1p-52;
    if (ep_mlp > ep) ep = ep_mlp;
  }
  Bounds b;
  // R32 = fl(R^) with R^ = L1^2 / S2 evaluated in double-float (2^-40) from
  // sums within relative g: R32 / R within (1 + g)^2 / (1 - g) (1 + 2^-40) (1 + u);
  // 2^-30 covers subnormal squares (S2 >= 2^-100).
  b.rho_r = (1.0 + g) * (1.0 + g) / (1.0 - g) * (1.0 + 0x1p-40) * (1.0 + u) - 1.0 + 0x1p-30;
  // s32 = fl(s^) with s^ = P / (sqrt(A) sqrt(B)) in double-float: A and B
  // within g contribute g (half each through the roots), the double-float
  // operations 2^-40, the final rounding u, P's residue e_p sqrt(A B) an
  // absolute term; 2^-34 covers underflowed squares and products when
  // A, B >= 2^-100.
  b.es_rel = 1.02 * (g / (1.0 - g) + u + 0x1p-40 + 0x1p-34);
  b.es_abs = 1.02 * (ep / (1.0 - g)) + 0x1p-34;
  // float factors: rounding a double to float moves it by at most 2^-24
  // relative, so widening by 2^-22 before the cast keeps each one outward.
  b.r_lo = (float)((1.0 / (1.0 + b.rho_r)) * (1.0 - 0x1p-22));
  b.r_hi = (float)((1.0 / (1.0 - b.rho_r)) * (1.0 + 0x1p-22));
  b.s_abs = (float)(b.es_abs * (1.0 + 0x1p-22));
  b.s_rel = (float)(b.es_rel * (1.0 + 0x1p-22));
  // Double-float tier.  A group of at least 128 threads recomputes a row:
  // each thread adds its k terms per sum (k = its 16-byte chunks times the
  // elements per chunk, doubled for fp32, whose squares and products enter as
  // TwoProd pairs) into a double-float by TwoSum, so hi + (the exact errors)
  // is the exact partial sum and only the low part's additions round: at most
  // k^2 u^2 of the sum of |terms| T.  Merging two partials (TwoSum of the high
  // parts, two low-part additions) rounds by at most (2 j + 1) u^2 T at a
  // merge whose inputs carry low parts below j u T: the five shuffle levels
  // inside a warp add at most (10 k + 35) u^2 T, and merging at most 16 warp
  // partials in turn at most 15 (2 k + 43) u^2 T; in all
  // (k^2 + 40 k + 680) u^2 T <= 4 (k + 16)^2 u^2 T.  For L1, S2, A, B, T is
  // the sum itself; for P, T = sum |x'x''| <= sqrt(A B).  Keys then: R from
  // L1^2 / S2 within (1 + e)^2 / (1 - e) (1 + 2^-40) of the truth, s within
  // e + |s| (e + 2^-40), the double-float operations' 2^-40 covering their
  // own roundings.
  const int per_chunk_df = 16 / elem_bytes(dtype);
  const double chunks_df = (double)((d / per_chunk_df + 127) / 128);
  const double k_df = chunks_df * per_chunk_df * (dtype == TR_F32 ? 2.0 : 1.0);
  const double e_df = 4.0 * (k_df + 16.0) * (k_df + 16.0) * u * u;
  const double r_df = (1.0 + e_df) * (1.0 + e_df) / (1.0 - e_df) * (1.0 + 0x1p-40) - 1.0;
  b.df_r = (float)(1.05 * r_df / (1.0 - r_df));  // relative to R_df
  b.df_s_abs = (float)(1.05 * e_df / (1.0 - e_df) + 0x1p-60);
  b.df_s_rel = (float)(1.05 * (e_df + 0x1p-40));
  return b;
}

// Sums below kTiny or above kHuge (or non-finite) are outside the fp32 error
// model above (underflow, overflow): such rows are settled exactly.
constexpr float kTiny = 0x1p-100f;
constexpr float kHuge = 0x1p+100f;

// ---------------------------------------------------------------- workspace
inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// [stats: total x TR_STATS_WORDS fp32][exact records: total x ExactRec]
struct WsLayout {
  size_t stats, exact, total;
};
inline WsLayout ws_layout(long long total_rows) {
  WsLayout w;
  w.stats = 0;
  w.exact = align_up(w.stats + (size_t)total_rows * TR_STATS_WORDS * sizeof(float), 256);
  w.total = align_up(w.exact + (size_t)total_rows * sizeof(ExactRec), 256);
  return w;
}

// ---------------------------------------------------------------- launch order
// Programmatic dependent launch: a kernel launched with pdl = true may be
// scheduled while the kernel before it on the stream still runs, once every
// CTA of that kernel has called pdl_trigger() (or exited); it calls
// pdl_wait() before it reads anything that kernel writes (the wait returns
// at once after a normal launch).  This hides the launch of a kernel behind
// the tail of the one before it: the single-call entry points use it, the
// pipeline does not (there a waiting grid would hold SMs that the next
// batch's scoring needs).
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... P, typename... A>
cudaError_t launch_kernel(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                          A &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<A>(args)...);
}

// ---------------------------------------------------------------- launchers
struct SelectArgs {
  const void *x, *x_pre, *x_post;
  int dtype, d, batch, n_uniform;
  const int32_t *cu_seqlens;
  const float *stats;
  const int32_t *k, *k1, *cu_k;
  int32_t *idx;
  uint8_t *role;      // or NULL
  float *h2, *s;      // exact fix-ups, or NULL
  ExactRec *exact;    // [total] scratch
  int32_t *status;    // or NULL
  Bounds bounds;
  int max_n;
  long long total_rows;  // rows of x, x', x'' and of the statistics
  bool stride_interval;  // diversity picks at floor(j M / K2) instead of j t
};

size_t select_smem_bytes(int max_n);  // dynamic shared memory of one select CTA
cudaError_t launch_score(const void *x, const void *x_pre, const void *x_post, int dtype, int d, long long total,
                         float *stats, float *h2, float *s, cudaStream_t st);
// max_ctas > 0 caps the grid (each CTA then selects several images in turn);
// pdl: programmatic dependent launch after the kernel before it on st.
cudaError_t launch_select(const SelectArgs &a, cudaStream_t st, int max_ctas, bool pdl);
int sm_count();  // SMs of the current device (cached), 0 on error
cudaError_t launch_select_gather(const SelectArgs &a, void *y, cudaStream_t st, bool pdl);
cudaError_t launch_gather(const void *x, long long total_rows, int dtype, int d, int batch, int n_uniform,
                          const int32_t *cu_seqlens, const int32_t *cu_k, const int32_t *idx, int total_k, void *y,
                          cudaStream_t st, bool pdl);

}  // namespace tr
