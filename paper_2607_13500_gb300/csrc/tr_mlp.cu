// The vision encoder's final-layer MLP, x'' = W2 sigma(W1 x') (Eq. 5), on
// the 5th-generation tensor cores, with ALTR's token scoring (Eq. 3-4 and
// Eq. 6) fused into the epilogue of its second GEMM.
//
// The paper takes x' and x'' from the encoder's forward pass "at no extra
// cost" (Section IV-B).  Here the second GEMM's epilogue, which produces
// x'' anyway, rounds each element to bf16, stores it, forms the block
// output x = bf16(resid + x'') and accumulates the five row sums of the
// selection -- L1 = sum|x|, S2 = sum x^2, A = sum x'^2, B = sum x''^2,
// P = sum x'x'' -- from the stored values, so a separate scoring pass over
// x, x', x'' is not needed and the selection stays a function of the stored
// tensors.  The row records it writes are the ones tr_score writes.
//
// One kernel serves both GEMMs (C[m, n] = A[m, k] B[n, k]^T, bf16 operands,
// fp32 accumulation): a persistent grid of one CTA per SM walks 128 x 256
// output tiles (tile t: row block t / n_tiles, column block t % n_tiles,
// so the CTAs running at one time share row blocks of A in L2).  Per CTA:
//   warp 0      TMA producer: A and B k-blocks (64 wide, 128-byte swizzle)
//               into a 4-stage shared-memory ring;
//   warp 1      allocates 512 TMEM columns (two 128 x 256 fp32
//               accumulators) and issues tcgen05.mma (M 128, N 256, K 16)
//               from one thread, committing each stage back to the
//               producer and each finished accumulator to the epilogue;
//   warps 2-    epilogue: one thread per accumulator row (TMEM lane: a
//               warp reads the lane quarter warp % 4) and column part, 16
//               columns per tcgen05.ld.  The score GEMM runs 8 warps (2-9,
//               column halves): it stores x'' and x and accumulates the row
//               sums.  The hidden GEMM runs 16 (2-17, column quarters):
//               bias + activation, and H through TMA stores of 32 x 32
//               blocks; the projector 8 (halves, 32 x 64 blocks).
// The projector mode (tr_project_kept) is the hidden GEMM with its A rows
// gathered: A row j is token idx[j] of the image that owns kept slot j, so
// the first projector layer reads X* = X_imp union X_div (Eq. 7) straight
// from x without a gathered copy.  Four more warps (10-13) bring those
// rows: lanes 0-7 of each load four rows of each A k-block with one TMA
// tile::gather4 load (four 64-element rows of x by index, one-row box,
// 128-byte swizzle -- the rows land in the layout the tensor cores read: the
// swizzle follows the shared-memory address); a group with a row past the
// kept slots (or a k-block past x's columns) takes four one-row tiled loads
// instead, an outside row at coordinate -1, which reads zeros.  Each loader
// warp's lane 0 adds its rows' bytes to the stage's transaction count and
// arrives once.  The rate at which one warp issues TMA loads sets the pace:
// 128 one-row loads per stage took 769 us from one warp and 273 us from
// four, the gather4 loads 314 us from one warp and 200 us from four.  The
// same layer on the gathered copy (tr_project: the hidden mode, plain tile
// loads) is faster -- 86 us against 182 us on 12288 kept rows, 1024 -> 4096,
// plus 12 us for the gather that writes the copy -- and gives the same z.
//
// The epilogue of tile i overlaps the main loop of tile i + 1 (two TMEM
// accumulators), but not for free: epilogue arithmetic on the SM
// sub-partitions that also hold the producer and MMA warps slows the main
// loop.  In a modified copy of the score GEMM with the sums' arithmetic
// skipped on sub-partitions 0-1 it took 224 us, on 2-3 254 us, on all four
// 193 us, against 257 us with none skipped.  So the epilogues do their fp32
// arithmetic on packed pairs (add / mul / fma.f32x2, one instruction per two
// columns): 6-7 % off all three modes.  A row's sums over its 2 n_tiles
// column halves are combined by the last of the warps that worked on them
// (an arrival counter; no warp or CTA waits for another), in column order,
// so the record does not depend on which finished first.
#include <cuda.h>
#include <cuda_bf16.h>

#include <atomic>
#include <climits>
#include <mutex>

#include "tr_internal.cuh"
#include "tr_record.cuh"
#include "tr_tc.cuh"

namespace tr {
namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64, kStages = 4;
constexpr int kATile = kBM * kBK * 2;             // bytes of one A k-block
constexpr int kBTile = kBN * kBK * 2;             // bytes of one B k-block
constexpr int kStageBytes = kATile + kBTile;      // 48 KiB
constexpr int kEpiWarps = 8;                      // score mode: two warpgroups, column halves of a tile
enum { kModeHidden = 0, kModeScore = 1, kModeProject = 2 };
// Epilogue warps per mode: the hidden GEMM's epilogue (activation and a TMA
// store) runs four warpgroups, one per column quarter, so that more warps
// hide the latencies of its TMEM loads and activation arithmetic; the score
// and projector epilogues run two (column halves) -- the projector's
// threads also include its four row-loader warps (measured on clip_mlp576's
// projector: four loader warps with 8 epilogue warps 200 us, with 16 195 us
// but spilling; two loader warps with 16, 226 us; eight with 8, 212 us).
__host__ __device__ constexpr int epi_warps(int mode) { return mode == kModeHidden ? 2 * kEpiWarps : kEpiWarps; }
__host__ __device__ constexpr int epi_parts(int mode) { return epi_warps(mode) / 4; }  // column parts of a tile
// producer, MMA issuer, epilogue (+ the A-row loader warps of the projector mode)
constexpr int kLoadRows = 4;   // projector: rows per loader lane and k-block, one tile::gather4
constexpr int kLoadWarps = 4;  // projector: loader warps, kBM / (kLoadRows kLoadWarps) lanes each
constexpr int kLoadLanes = kBM / (kLoadRows * kLoadWarps);
static_assert(kLoadLanes * kLoadRows * kLoadWarps == kBM && kLoadLanes <= 32, "the loaders cover a tile's rows");
__host__ __device__ constexpr int gemm_threads(int mode) {
  return 64 + 32 * epi_warps(mode) + (mode == kModeProject ? 32 * kLoadWarps : 0);
}
constexpr int kTmemCols = 2 * kBN;                // two accumulators
constexpr int kChunk = 16;                        // columns per tcgen05.ld
constexpr int kPartWords = 10;                    // hi, lo of L1, S2, A, B, P
constexpr uint32_t kIdesc = tc::idesc_bf16(kBM, kBN);
// Per epilogue warp of the hidden and projector modes, a 32-row bf16 output
// block staged for a TMA store: 32 columns (64-byte rows, 64-byte swizzle)
// with four column parts, 64 (128-byte rows and swizzle) with two; 32 KiB in
// all either way.
constexpr int kStageOutAll = 32 * 1024;
__host__ __device__ constexpr int stage_out(int mode) { return kStageOutAll / epi_warps(mode); }
constexpr size_t kGemmSmem = (size_t)kStages * kStageBytes + kStageOutAll + 1024 + 256;

struct GemmArgs {
  int m, n, k;          // C[m, n] = A[m, k] B[n, k]^T
  int n_tiles, tiles, kblocks;
  const float *bias;    // [n] or NULL
  int act;              // hidden GEMM: TR_ACT_*
  uint16_t *out;        // hidden: H [m, n]; score: x'' [m, n] (bf16 bits)
  const uint16_t *x_pre, *resid;  // score: x' [m, n], residual [m, n] or NULL
  uint16_t *x;          // score: block output [m, n]
  float *part;          // score: [row blocks][n_tiles][2 halves][4][kPartWords][32] partial sums
  int *arrivals;        // score: [row blocks][4], zero at launch
  float4 *stats;        // score: [m] records (two float4 each)
  float *h2, *s;        // score: optional outputs
  int32_t *err;         // optional: set when a pipeline wait timed out
  // projector mode: A row j = x[first row of the image owning kept slot j + idx[j]]
  const uint16_t *gx;   // x [total_rows, k]
  long long total_rows;
  int batch, n_uniform;
  const int32_t *cu_seqlens, *cu_k, *idx;
};

__device__ __forceinline__ float bf16_val(uint32_t bits16) { return __uint_as_float(bits16 << 16); }

// 2^x and 1/x by the hardware approximations (PTX ex2.approx, rcp.approx:
// relative error about 2^-22 and 2^-23), a few fp32 ulp, far inside the bf16
// rounding of the activations below.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32 pairs (one instruction for two lanes of arithmetic, each
// rounded to nearest like its scalar form).
__device__ __forceinline__ float2 f2(float v) { return make_float2(v, v); }
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {  // a - b, one rounding
  return __ffma2_rn(b, f2(-1.f), a);
}
__device__ __forceinline__ float2 ex2_2(float2 x) { return make_float2(ex2_approx(x.x), ex2_approx(x.y)); }
__device__ __forceinline__ float2 rcp_2(float2 x) { return make_float2(rcp_approx(x.x), rcp_approx(x.y)); }

// erf(z) for z >= 0 by Abramowitz and Stegun, Handbook of Mathematical
// Functions (1964), formula 7.1.26: 1 - (a1 t + ... + a5 t^5) exp(-z^2) with
// t = 1 / (1 + p z), |error| <= 1.5e-7; with the approximate exponential and
// reciprocal GELU below stays within ~2e-7 |v| of x Phi(x), far inside the
// bf16 rounding of its result.  Two arguments at a time.
__device__ __forceinline__ float2 erf_as2(float2 z) {
  const float2 t = rcp_2(__ffma2_rn(z, f2(0.3275911f), f2(1.f)));
  float2 poly = __ffma2_rn(t, f2(1.061405429f), f2(-1.453152027f));
  poly = __ffma2_rn(t, poly, f2(1.421413741f));
  poly = __ffma2_rn(t, poly, f2(-0.284496736f));
  poly = __ffma2_rn(t, poly, f2(0.254829592f));
  poly = __fmul2_rn(t, poly);
  const float2 ez = ex2_2(__fmul2_rn(__fmul2_rn(z, z), f2(-1.4426950408889634f)));  // exp(-z^2)
  return sub2(f2(1.f), __fmul2_rn(poly, ez));
}

// The activation sigma of the hidden layer (and the projector) on a pair of
// pre-activations.
__device__ __forceinline__ float2 activate2(float2 v, int act) {
  if (act == TR_ACT_GELU) {  // v Phi(v) = v (1 + erf(v / sqrt 2)) / 2
    const float2 e = erf_as2(__fmul2_rn(make_float2(fabsf(v.x), fabsf(v.y)), f2(0.70710678118654752f)));
    return __fmul2_rn(__fmul2_rn(v, f2(0.5f)), __fadd2_rn(f2(1.f), make_float2(copysignf(e.x, v.x), copysignf(e.y, v.y))));
  }
  if (act == TR_ACT_QUICK_GELU) {  // v sigma(1.702 v) = v / (1 + 2^(-1.702 log2(e) v)), the exponent capped
    float2 z = __fmul2_rn(v, f2(-2.4554669595930156f));
    z.x = fminf(z.x, 126.f);
    z.y = fminf(z.y, 126.f);
    return __fmul2_rn(v, rcp_2(__fadd2_rn(ex2_2(z), f2(1.f))));
  }
  return v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ void flag_error(const GemmArgs &g, int code) {
  if (g.err) atomicOr(g.err, code);
}

// Hidden GEMM epilogue for 16 columns of one row: H = bf16(act(acc + b1)).
__device__ __forceinline__ void epi_hidden(const GemmArgs &g, long long row, int col0, const float (&v)[16]) {
  float2 a[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) a[i] = make_float2(v[2 * i], v[2 * i + 1]);
  if (g.bias) {  // the same 16 values in every lane: four broadcast loads
    const float4 *bp = reinterpret_cast<const float4 *>(g.bias + col0);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float4 b = __ldg(bp + i);
      a[2 * i] = __fadd2_rn(a[2 * i], make_float2(b.x, b.y));
      a[2 * i + 1] = __fadd2_rn(a[2 * i + 1], make_float2(b.z, b.w));
    }
  }
  uint32_t w[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 h = activate2(a[i], g.act);
    w[i] = pack_bf16x2(h.x, h.y);
  }
  uint4 *dst = reinterpret_cast<uint4 *>(g.out + row * g.n + col0);
  dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
  dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
}

// The 16 columns of x' and of the residual that the score epilogue of one
// chunk reads, loaded one chunk ahead of their use.
struct ScoreIn {
  uint4 p0, p1, r0, r1;
};
__device__ __forceinline__ void load_score_in(const GemmArgs &g, long long row, int col0, ScoreIn &in) {
  const long long base = row * g.n + col0;
  const uint4 *pp = reinterpret_cast<const uint4 *>(g.x_pre + base);
  in.p0 = __ldg(pp);
  in.p1 = __ldg(pp + 1);
  if (g.resid) {
    const uint4 *rp = reinterpret_cast<const uint4 *>(g.resid + base);
    in.r0 = __ldg(rp);
    in.r1 = __ldg(rp + 1);
  } else {
    in.r0 = in.r1 = make_uint4(0u, 0u, 0u, 0u);
  }
}

// The score epilogue keeps its five double-float sums as fp32 pairs:
// component x takes the even columns, component y the odd ones, merged once
// per tile.
__device__ __forceinline__ float2 bf16x2_f2(uint32_t w) {  // the two bf16 of a word as fp32
  return make_float2(bf16_val(w & 0xffffu), bf16_val(w >> 16));
}
struct DF2 {
  float2 hi, lo;
};
struct Acc2 {
  DF2 l1, s2, a, b, p;
};
// acc += v with Knuth's TwoSum per component: s = hi + v, and the rounding
// error (hi - (s - (s - hi))) + (v - (s - hi)) joins lo.  With nb = hi - s
// (= -(s - hi) exactly, rounding being symmetric) the steps are the scalar
// df_add's, two lanes at a time.
__device__ __forceinline__ void df2_add(DF2 &acc, float2 v) {
  const float2 s = __fadd2_rn(acc.hi, v);
  const float2 nb = sub2(acc.hi, s);
  const float2 aa = __fadd2_rn(s, nb);
  acc.lo = __fadd2_rn(acc.lo, __fadd2_rn(sub2(acc.hi, aa), __fadd2_rn(v, nb)));
  acc.hi = s;
}
// acc += u v for products exact in fp32 (bf16 times bf16): the fused
// multiply-add rounds hi + u v once, as the sum of the exact product would.
__device__ __forceinline__ void df2_add_prod(DF2 &acc, float2 u, float2 v) {
  const float2 s = __ffma2_rn(u, v, acc.hi);
  const float2 nb = sub2(acc.hi, s);
  const float2 aa = __fadd2_rn(s, nb);
  acc.lo = __fadd2_rn(acc.lo, __fadd2_rn(sub2(acc.hi, aa), __ffma2_rn(u, v, nb)));
  acc.hi = s;
}
__device__ __forceinline__ void df2_fold(DF &out, const DF2 &in) {  // even + odd columns
  out.hi = in.hi.x;
  out.lo = in.lo.x;
  df_merge(out, in.hi.y, in.lo.y);
}

// Score GEMM epilogue for 16 columns of one row: x'' = bf16(acc + b2),
// x = bf16(resid + x''), both stored; the five sums take the stored values
// (products and squares of bf16 values are exact in fp32; each term enters
// its double-float sum through TwoSum).
__device__ __forceinline__ void epi_score(const GemmArgs &g, long long row, int col0, const float (&v)[16],
                                          const ScoreIn &in, Acc2 &acc) {
  const long long base = row * g.n + col0;
  const uint32_t pw[8] = {in.p0.x, in.p0.y, in.p0.z, in.p0.w, in.p1.x, in.p1.y, in.p1.z, in.p1.w};
  const uint32_t rw[8] = {in.r0.x, in.r0.y, in.r0.z, in.r0.w, in.r1.x, in.r1.y, in.r1.z, in.r1.w};
  float2 a[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) a[i] = make_float2(v[2 * i], v[2 * i + 1]);
  if (g.bias) {
    const float4 *bp = reinterpret_cast<const float4 *>(g.bias + col0);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float4 b = __ldg(bp + i);
      a[2 * i] = __fadd2_rn(a[2 * i], make_float2(b.x, b.y));
      a[2 * i + 1] = __fadd2_rn(a[2 * i + 1], make_float2(b.z, b.w));
    }
  }
  uint32_t qo[8], xo[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    qo[i] = pack_bf16x2(a[i].x, a[i].y);  // x''
    const float2 q = bf16x2_f2(qo[i]);
    if (g.resid) {
      const float2 xs = __fadd2_rn(bf16x2_f2(rw[i]), q);
      xo[i] = pack_bf16x2(xs.x, xs.y);
    } else {
      xo[i] = qo[i];
    }
    const float2 xa = bf16x2_f2(xo[i] & 0x7fff7fffu);  // |x|
    const float2 p = bf16x2_f2(pw[i]);                 // x'
    df2_add(acc.l1, xa);
    df2_add_prod(acc.s2, xa, xa);
    df2_add_prod(acc.a, p, p);
    df2_add_prod(acc.b, q, q);
    df2_add_prod(acc.p, p, q);
  }
  uint4 *dq = reinterpret_cast<uint4 *>(g.out + base);
  dq[0] = make_uint4(qo[0], qo[1], qo[2], qo[3]);
  dq[1] = make_uint4(qo[4], qo[5], qo[6], qo[7]);
  uint4 *dx = reinterpret_cast<uint4 *>(g.x + base);
  dx[0] = make_uint4(xo[0], xo[1], xo[2], xo[3]);
  dx[1] = make_uint4(xo[4], xo[5], xo[6], xo[7]);
}

// Score epilogue of one tile half for this warp: the 8 chunks of 16 columns
// of its column half, each chunk's TMEM load (and its x' and residual
// loads) issued while the chunk before it is processed.
//
// Hidden / projector epilogue of one of a tile's kParts column parts for
// this warp: chunks of 16 columns, H = bf16(act(acc + bias)), staged in this
// warp's 32-row block of kBlk = 64 / (kParts / 2) columns, whose rows are
// kBlk * 2 bytes with the swizzle of that span (unit u of row r at
// r * 2 kBlk + ((u ^ ((r / (8 / (kBlk / 8))) % (kBlk / 8))) << 4): the 32
// lanes' 16-byte writes take the fewest shared-memory wavefronts), and
// written by one TMA store per block, so global memory sees whole row
// segments.  The next chunk's TMEM load and bias are in flight while a chunk
// is processed; the block is rewritten only after its previous store has
// read it.  Rows and columns past the output are computed from zero operands
// and clipped by the store.
template <int kParts>
__device__ __forceinline__ void drain_tile_store(const GemmArgs &g, const CUtensorMap *map_out, uint32_t buf,
                                                 uint32_t taddr, int part, int nt, long long row0) {
  constexpr int kChunks = kBN / kParts / kChunk;  // 8 (halves) or 4 (quarters)
  constexpr int kBlk = 128 / kParts;              // block columns: 64 or 32
  constexpr int kUnits = kBlk / 8;                // 16-byte units per block row: 8 or 4
  constexpr int kPerBlk = kBlk / kChunk;          // chunks per block: 4 or 2
  const int lane = threadIdx.x & 31;
  const int col_first = nt * kBN + part * (kBN / kParts);
  int chunks = 0;
  while (chunks < kChunks && col_first + chunks * kChunk < g.n) ++chunks;
  if (chunks == 0) return;
  uint32_t cur[16], nxt[16];
  float4 bc[4];
  auto load_bias = [&](int col0, float4 (&b)[4]) {
    if (g.bias) {
      const float4 *bp = reinterpret_cast<const float4 *>(g.bias + col0);
#pragma unroll
      for (int i = 0; i < 4; ++i) b[i] = __ldg(bp + i);
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) b[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  const uint32_t tcol = taddr + (uint32_t)(part * (kBN / kParts));
  tc::tmem_ld16_issue(tcol, cur);
  tc::tmem_ld_wait(cur);
  const uint32_t rowbuf = buf + (uint32_t)(lane * kBlk * 2);
  const uint32_t sw = (uint32_t)((lane / (8 / kUnits)) % kUnits);  // the swizzle's row term
  for (int c = 0; c < chunks; ++c) {
    const int col0 = col_first + c * kChunk;
    const bool more = c + 1 < chunks;
    if (more) tc::tmem_ld16_issue(tcol + (uint32_t)((c + 1) * kChunk), nxt);
    load_bias(col0, bc);  // the same 16 values in every lane (broadcast loads, cached)
    const float bias[16] = {bc[0].x, bc[0].y, bc[0].z, bc[0].w, bc[1].x, bc[1].y, bc[1].z, bc[1].w,
                            bc[2].x, bc[2].y, bc[2].z, bc[2].w, bc[3].x, bc[3].y, bc[3].z, bc[3].w};
    uint32_t w[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float2 h = activate2(__fadd2_rn(make_float2(__uint_as_float(cur[2 * i]), __uint_as_float(cur[2 * i + 1])),
                                            make_float2(bias[2 * i], bias[2 * i + 1])),
                                 g.act);
      w[i] = pack_bf16x2(h.x, h.y);
    }
    if (c % kPerBlk == 0 && c > 0) {  // the block's previous store must have read it
      if (lane == 0) tc::bulk_wait_read();
      __syncwarp();
    }
    const uint32_t u = 2u * (uint32_t)(c % kPerBlk);
    tc::st_shared_v4(rowbuf + ((u ^ sw) << 4), w[0], w[1], w[2], w[3]);
    tc::st_shared_v4(rowbuf + (((u + 1u) ^ sw) << 4), w[4], w[5], w[6], w[7]);
    if (c % kPerBlk == kPerBlk - 1 || !more) {  // a block is complete: one TMA store for the warp's 32 rows
      tc::fence_async_shared();
      __syncwarp();
      if (lane == 0 && row0 < g.m) {  // a block wholly past the last row is not stored
        tc::tma_store_2d(map_out, col_first + kBlk * (c / kPerBlk), (int)row0, buf);
        tc::bulk_commit();
      }
    }
    if (more) {
      tc::tmem_ld_wait(nxt);
#pragma unroll
      for (int i = 0; i < 16; ++i) cur[i] = nxt[i];
    }
  }
  if (lane == 0) tc::bulk_wait_read();  // the block may be rewritten by the next tile
  __syncwarp();
}

template <int kMode>
__device__ __forceinline__ void drain_tile(const GemmArgs &g, uint32_t taddr, int half, int nt, long long row,
                                           bool row_ok, Acc &sums) {
  constexpr int kChunks = kBN / 2 / kChunk;
  int chunks = 0;  // chunks of this half inside the output (uniform across the warp)
  while (chunks < kChunks && nt * kBN + half * (kBN / 2) + chunks * kChunk < g.n) ++chunks;
  if (chunks == 0) return;
  uint32_t cur[16], nxt[16];
  ScoreIn in_cur{}, in_nxt{};
  Acc2 acc2{};
  const int col_first = nt * kBN + half * (kBN / 2);
  tc::tmem_ld16_issue(taddr + (uint32_t)(half * (kBN / 2)), cur);
  if (kMode == kModeScore && row_ok) load_score_in(g, row, col_first, in_cur);
  tc::tmem_ld_wait(cur);
  for (int c = 0; c < chunks; ++c) {
    const int col0 = col_first + c * kChunk;
    const bool more = c + 1 < chunks;
    if (more) {
      tc::tmem_ld16_issue(taddr + (uint32_t)(half * (kBN / 2) + (c + 1) * kChunk), nxt);
      if (kMode == kModeScore && row_ok) load_score_in(g, row, col0 + kChunk, in_nxt);
    }
    if (row_ok) {
      float v[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(cur[i]);
      if (kMode == kModeScore)
        epi_score(g, row, col0, v, in_cur, acc2);
      else
        epi_hidden(g, row, col0, v);
    }
    if (more) {
      tc::tmem_ld_wait(nxt);
#pragma unroll
      for (int i = 0; i < 16; ++i) cur[i] = nxt[i];
      in_cur = in_nxt;
    }
  }
  if (kMode == kModeScore) {
    df2_fold(sums.l1, acc2.l1);
    df2_fold(sums.s2, acc2.s2);
    df2_fold(sums.a, acc2.a);
    df2_fold(sums.b, acc2.b);
    df2_fold(sums.p, acc2.p);
  }
}

// This warp's 32 rows of one tile half are done: publish their partial
// sums; the warp that completes a row block's quadrant (the last of its
// 2 n_tiles column halves to arrive) merges the partials in column order
// and writes the rows' records.
__device__ __forceinline__ long long part_slot(const GemmArgs &g, int rb, int nt, int half, int q) {
  return (((long long)(rb * g.n_tiles + nt) * 2 + half) * 4 + q) * (kPartWords * 32);
}
__device__ __forceinline__ void publish_rows(const GemmArgs &g, int rb, int nt, int half, int q, long long row,
                                             bool row_ok, const Acc &acc) {
  const int lane = threadIdx.x & 31;
  float *dst = g.part + part_slot(g, rb, nt, half, q) + lane;
  const float vals[kPartWords] = {acc.l1.hi, acc.l1.lo, acc.s2.hi, acc.s2.lo, acc.a.hi,
                                  acc.a.lo,  acc.b.hi,  acc.b.lo,  acc.p.hi,  acc.p.lo};
#pragma unroll
  for (int j = 0; j < kPartWords; ++j) __stcg(dst + 32 * j, vals[j]);
  __threadfence();
  __syncwarp();
  int last = 0;
  if (lane == 0) last = atomicAdd(g.arrivals + rb * 4 + q, 1) == 2 * g.n_tiles - 1;
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence();
  Acc tot{{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
  for (int t = 0; t < 2 * g.n_tiles; ++t) {
    const float *src = g.part + part_slot(g, rb, t >> 1, t & 1, q) + lane;
    float w[kPartWords];
#pragma unroll
    for (int j = 0; j < kPartWords; ++j) w[j] = __ldcg(src + 32 * j);
    df_merge(tot.l1, w[0], w[1]);
    df_merge(tot.s2, w[2], w[3]);
    df_merge(tot.a, w[4], w[5]);
    df_merge(tot.b, w[6], w[7]);
    df_merge(tot.p, w[8], w[9]);
  }
  if (row_ok) write_record(tot, row, g.stats, g.h2, g.s);
  if (lane == 0) g.arrivals[rb * 4 + q] = 0;  // ready for the next launch
}

// Row of x that kept slot j names (projector mode), or -1: the image b with
// cu_k[b] <= j < cu_k[b + 1], its local index idx[j] checked against the
// image's tokens (an index outside them gives a zero row, never another
// image's token or an address outside x).
__device__ __forceinline__ long long kept_source_row(const GemmArgs &g, long long j) {
  if (j >= g.m) return -1;
  int lo = 0, hi = g.batch;  // cu_k[lo] <= j < cu_k[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(g.cu_k + mid) <= j) lo = mid; else hi = mid;
  }
  const long long first = g.cu_seqlens ? (long long)__ldg(g.cu_seqlens + lo) : (long long)lo * g.n_uniform;
  const long long n_b = g.cu_seqlens ? (long long)__ldg(g.cu_seqlens + lo + 1) - first : (long long)g.n_uniform;
  const int local = __ldg(g.idx + j);
  if (local < 0 || local >= n_b || first < 0 || first + local >= g.total_rows) return -1;
  return first + local;
}

template <int kMode>
__global__ void __launch_bounds__(gemm_threads(kMode), 1)
    k_mlp_gemm(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
               const __grid_constant__ CUtensorMap map_out, const GemmArgs g) {
  extern __shared__ unsigned char smem_raw[];
  // stage tiles at a 1024-byte boundary (the swizzle atom), barriers after them
  unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                          ~static_cast<uintptr_t>(1023));
  const uint32_t out_stage = tc::smem_u32(smem + (size_t)kStages * kStageBytes);  // epilogue staging
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)kStages * kStageBytes + kStageOutAll);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * kStages + 5);
  const uint32_t sbase = tc::smem_u32(smem);
  const uint32_t b0 = tc::smem_u32(bars);
  auto full = [&](int s) { return b0 + 8u * s; };
  auto empty = [&](int s) { return b0 + 8u * (kStages + s); };
  auto tfull = [&](int a) { return b0 + 8u * (2 * kStages + a); };
  auto tempty = [&](int a) { return b0 + 8u * (2 * kStages + 2 + a); };
  const uint32_t done = b0 + 8u * (2 * kStages + 4);
  auto sa = [&](int s) { return sbase + (uint32_t)(s * kStageBytes); };
  auto sb = [&](int s) { return sbase + (uint32_t)(s * kStageBytes + kATile); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(full(s), kMode == kModeProject ? 1 + kLoadWarps : 1);  // + one arrival per loader warp
      tc::mbar_init(empty(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(tfull(a), 1);
      tc::mbar_init(tempty(a), 32 * epi_warps(kMode));
    }
    tc::mbar_init(done, 1);
    tc::mbar_fence_init();
    tc::tma_prefetch_map(&map_a);
    tc::tma_prefetch_map(&map_b);
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(tmem_slot), kTmemCols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    int stage = 0;
    uint32_t phase = 0, filled = 0, last_parity = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < g.tiles && ok; tile += gridDim.x) {
      const int rb = tile / g.n_tiles, nt = tile - rb * g.n_tiles;
      for (int kb = 0; kb < g.kblocks; ++kb) {
        if (!tc::mbar_wait_warp(empty(stage), phase ^ 1u)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          if (kMode == kModeProject) {  // A comes from the row loaders
            tc::mbar_expect_tx(full(stage), kBTile);
          } else {
            tc::mbar_expect_tx(full(stage), kStageBytes);
            tc::tma_load_2d(sa(stage), &map_a, kb * kBK, rb * kBM, full(stage));
          }
          tc::tma_load_2d(sb(stage), &map_b, kb * kBK, nt * kBN, full(stage));
        }
        __syncwarp();
        filled |= 1u << stage;
        last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) flag_error(g, 1);
    // the loads already issued land before the CTA may exit
    for (int s = 0; s < kStages; ++s)
      if (filled & (1u << s)) tc::mbar_wait_warp(full(s), (last_parity >> s) & 1u);
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    int stage = 0, acc = 0;
    uint32_t phase = 0, acc_phase = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < g.tiles && ok; tile += gridDim.x) {
      if (!tc::mbar_wait_warp(tempty(acc), acc_phase ^ 1u)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      const uint32_t d = tmem + (uint32_t)(acc * kBN);
      for (int kb = 0; kb < g.kblocks; ++kb) {
        if (!tc::mbar_wait_warp(full(stage), phase)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        if (lane == 0) {
          const uint64_t da = tc::sw128_desc(sa(stage)), db = tc::sw128_desc(sb(stage));
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)  // 32 bytes further along K per step (start address >> 4: + 2)
            tc::mma_bf16(d, da + 2u * k, db + 2u * k, kIdesc, (kb | k) != 0);
          tc::mma_commit(empty(stage));  // the stage is free once these MMAs have read it
        }
        __syncwarp();
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      if (lane == 0) tc::mma_commit(tfull(acc));  // the accumulator is complete
      __syncwarp();
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (!ok && lane == 0) flag_error(g, 2);
    // every MMA issued has completed before TMEM is released
    if (lane == 0) tc::mma_commit(done);
    __syncwarp();
    tc::mbar_wait_warp(done, 0);
  } else if (kMode == kModeProject && warp >= 2 + epi_warps(kMode)) {
    // ---------------------------------------------------------------- A rows (projector mode)
    // lane l < kLoadLanes of loader warp w brings rows 4 j .. 4 j + 3 (j = w
    // kLoadLanes + l) of each A k-block with one tile::gather4 load; a group
    // with a row outside x (past the kept slots) or a k-block past x's
    // columns takes four one-row loads instead, an outside row at coordinate
    // -1, which reads zeros
    const int j = (warp - 2 - epi_warps(kMode)) * kLoadLanes + lane;
    const bool loads = lane < kLoadLanes;
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < g.tiles && ok; tile += gridDim.x) {
      const int rb = tile / g.n_tiles;
      int srow[kLoadRows];
      bool whole = true;
#pragma unroll
      for (int i = 0; i < kLoadRows; ++i) {
        const long long src = loads ? kept_source_row(g, (long long)rb * kBM + kLoadRows * j + i) : -1;
        srow[i] = src >= 0 ? (int)src : -1;
        whole &= src >= 0;
      }
      for (int kb = 0; kb < g.kblocks; ++kb) {
        if (!tc::mbar_wait_warp(empty(stage), phase ^ 1u)) {
          ok = false;
          break;
        }
        if (lane == 0) tc::mbar_expect_tx(full(stage), kATile / kLoadWarps);  // this warp's rows; one arrival
        __syncwarp();
        const uint32_t dst = sa(stage) + (uint32_t)(kLoadRows * j * kBK * 2);
        if (loads) {
          if (whole && (kb + 1) * kBK <= g.k) {  // rows and columns inside x
            tc::tma_gather4(dst, &map_a, kb * kBK, srow[0], srow[1], srow[2], srow[3], full(stage));
          } else {
#pragma unroll
            for (int i = 0; i < kLoadRows; ++i)
              tc::tma_load_2d(dst + (uint32_t)(i * kBK * 2), &map_a, kb * kBK, srow[i], full(stage));
          }
        }
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) flag_error(g, 8);
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;            // TMEM lane quadrant this warp may read
    const int half = (warp - 2) >> 2;  // column half (score) or quarter (hidden, projector) of the tile
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < g.tiles; tile += gridDim.x) {
      const int rb = tile / g.n_tiles, nt = tile - rb * g.n_tiles;
      if (!tc::mbar_wait_warp(tfull(acc), acc_phase)) {
        if (lane == 0) flag_error(g, 4);
        break;
      }
      tc::fence_after_sync();
      const long long row = (long long)rb * kBM + 32 * q + lane;
      const bool row_ok = row < g.m;
      const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(acc * kBN);
      Acc sums{{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
      if (kMode == kModeScore)
        drain_tile<kMode>(g, taddr, half, nt, row, row_ok, sums);
      else
        drain_tile_store<epi_parts(kMode)>(g, &map_out, out_stage + (uint32_t)((warp - 2) * stage_out(kMode)), taddr,
                                           half, nt,
                         row - lane);
      tc::fence_before_sync();
      tc::mbar_arrive(tempty(acc));  // the MMA warp may refill this accumulator
      if (kMode == kModeScore) publish_rows(g, rb, nt, half, q, row, row_ok, sums);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (kMode != kModeScore && lane == 0) tc::bulk_wait();  // this warp's output stores have completed
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- the SM-pair kernel
// The same GEMM with tcgen05's 2-SM MMA: a cluster of two CTAs shares each
// 256 x 256 output tile (tile t: row block t / n_tiles of 256 rows).  CTA
// rank r loads A rows 128 r .. 128 r + 127 of the tile and B rows (output
// columns) 128 r .. 128 r + 127 into its own shared memory -- 32 KiB per
// k-block stage, six stages -- and both CTAs' loads complete on the even
// CTA's stage barrier.  The even CTA alone issues the pair's MMAs (M 256,
// N 256, K 16), which read both CTAs' stages and write each CTA's 128
// accumulator rows into its own TMEM; its commits reach the same barriers
// in both CTAs (multicast).  Each CTA's epilogue drains its own rows and
// releases the accumulator on the even CTA's barrier.  Per SM a k-block
// brings 32 KiB of operands for a 128 x 256 x 64 product, against 48 KiB on
// one SM, so six stages in flight hide the load latency that four did not.
constexpr int kStagesP = 6;
constexpr int kHalfTile = 128 * kBK * 2;          // 128 rows of a k-block (A or B)
constexpr int kStagePBytes = 2 * kHalfTile;       // this CTA's A rows + B rows
constexpr uint32_t kIdescPair = tc::idesc_bf16(2 * kBM, kBN);
constexpr size_t kGemmPSmem = (size_t)kStagesP * kStagePBytes + kStageOutAll + 1024 + 256;

template <int kMode>
__global__ void __launch_bounds__(gemm_threads(kMode), 1)
    k_mlp_gemm_pair(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                    const __grid_constant__ CUtensorMap map_out, const GemmArgs g) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                          ~static_cast<uintptr_t>(1023));
  const uint32_t out_stage = tc::smem_u32(smem + (size_t)kStagesP * kStagePBytes);  // epilogue staging
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)kStagesP * kStagePBytes + kStageOutAll);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * kStagesP + 5);
  const uint32_t sbase = tc::smem_u32(smem);
  const uint32_t b0 = tc::smem_u32(bars);
  auto full = [&](int s) { return b0 + 8u * s; };
  auto empty = [&](int s) { return b0 + 8u * (kStagesP + s); };
  auto tfull = [&](int a) { return b0 + 8u * (2 * kStagesP + a); };
  auto tempty = [&](int a) { return b0 + 8u * (2 * kStagesP + 2 + a); };
  const uint32_t done = b0 + 8u * (2 * kStagesP + 4);
  auto sa = [&](int s) { return sbase + (uint32_t)(s * kStagePBytes); };
  auto sb = [&](int s) { return sbase + (uint32_t)(s * kStagePBytes + kHalfTile); };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = tc::cluster_rank();
  const bool leader = rank == 0;
  const int cluster = blockIdx.x >> 1, clusters = gridDim.x >> 1;
  // operand bytes landing on the even CTA's stage barrier per k-block (both CTAs)
  constexpr uint32_t kTx = kMode == kModeProject ? 2 * kHalfTile : 2 * kStagePBytes;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesP; ++s) {
      tc::mbar_init(full(s), kMode == kModeProject ? 1 + kLoadWarps : 1);  // + the even CTA's loader warps
      tc::mbar_init(empty(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(tfull(a), 1);
      tc::mbar_init(tempty(a), 2 * epi_warps(kMode));  // one arrival per epilogue warp of either CTA
    }
    tc::mbar_init(done, 1);
    tc::mbar_fence_init();
    tc::tma_prefetch_map(&map_a);
    tc::tma_prefetch_map(&map_b);
  }
  if (warp == 1) {
    tc::tmem_alloc_pair(tc::smem_u32(tmem_slot), kTmemCols);
    tc::tmem_relinquish_pair();
  }
  tc::fence_before_sync();
  tc::cluster_sync();  // barriers initialised and TMEM allocated in both CTAs
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;
  auto full_even = [&](int s) { return tc::map_shared(full(s), 0); };
  auto tempty_even = [&](int a) { return tc::map_shared(tempty(a), 0); };
  const int row_tiles = (g.m + 2 * kBM - 1) / (2 * kBM);
  const int tiles = row_tiles * g.n_tiles;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer (both CTAs)
    int stage = 0;
    uint32_t phase = 0, filled = 0, last_parity = 0;
    bool ok = true;
    for (int tile = cluster; tile < tiles && ok; tile += clusters) {
      const int rb = tile / g.n_tiles, nt = tile - rb * g.n_tiles;
      for (int kb = 0; kb < g.kblocks; ++kb) {
        if (!tc::mbar_wait_warp(empty(stage), phase ^ 1u)) {
          ok = false;
          break;
        }
        if (lane == 0) {
          const uint32_t bar = full_even(stage);
          if (leader) tc::mbar_expect_tx(full(stage), kTx);
          if (kMode != kModeProject)
            tc::tma_load_2d_pair(sa(stage), &map_a, kb * kBK, rb * 2 * kBM + (int)rank * kBM, bar);
          tc::tma_load_2d_pair(sb(stage), &map_b, kb * kBK, nt * kBN + (int)rank * 128, bar);
        }
        __syncwarp();
        filled |= 1u << stage;
        last_parity = (last_parity & ~(1u << stage)) | (phase << stage);
        if (++stage == kStagesP) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) flag_error(g, 1);
    // every load of either CTA lands on the even CTA's barriers: it waits for
    // them before the final cluster barrier, so no CTA exits with loads in flight
    if (leader)
      for (int s = 0; s < kStagesP; ++s)
        if (filled & (1u << s)) tc::mbar_wait_warp(full(s), (last_parity >> s) & 1u);
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer (even CTA)
    if (leader) {
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      for (int tile = cluster; tile < tiles && ok; tile += clusters) {
        if (!tc::mbar_wait_warp(tempty(acc), acc_phase ^ 1u)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t d = tmem + (uint32_t)(acc * kBN);
        for (int kb = 0; kb < g.kblocks; ++kb) {
          if (!tc::mbar_wait_warp(full(stage), phase)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
          if (lane == 0) {
            const uint64_t da = tc::sw128_desc(sa(stage)), db = tc::sw128_desc(sb(stage));
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              tc::mma_bf16_pair(d, da + 2u * k, db + 2u * k, kIdescPair, (kb | k) != 0);
            tc::mma_commit_pair(empty(stage), 0x3);  // both CTAs' stage is free once these MMAs read it
          }
          __syncwarp();
          if (++stage == kStagesP) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if (lane == 0) tc::mma_commit_pair(tfull(acc), 0x3);
        __syncwarp();
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok && lane == 0) flag_error(g, 2);
      if (lane == 0) tc::mma_commit_pair(done, 0x3);
      __syncwarp();
    }
    tc::mbar_wait_warp(done, 0);  // every pair MMA has completed (both CTAs' TMEM)
  } else if (kMode == kModeProject && warp >= 2 + epi_warps(kMode)) {
    // ---------------------------------------------------------------- A rows (projector mode)
    // as in the one-SM kernel, into this CTA's half of the pair's rows; the
    // loads land on the even CTA's barrier, whose loader warps expect both
    // CTAs' bytes (the odd CTA's loader warps do not arrive)
    const int j = (warp - 2 - epi_warps(kMode)) * kLoadLanes + lane;
    const bool loads = lane < kLoadLanes;
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int tile = cluster; tile < tiles && ok; tile += clusters) {
      const int rb = tile / g.n_tiles;
      int srow[kLoadRows];
      bool whole = true;
#pragma unroll
      for (int i = 0; i < kLoadRows; ++i) {
        const long long src =
            loads ? kept_source_row(g, (long long)rb * 2 * kBM + (long long)rank * kBM + kLoadRows * j + i) : -1;
        srow[i] = src >= 0 ? (int)src : -1;
        whole &= src >= 0;
      }
      for (int kb = 0; kb < g.kblocks; ++kb) {
        if (!tc::mbar_wait_warp(empty(stage), phase ^ 1u)) {
          ok = false;
          break;
        }
        if (lane == 0 && leader) tc::mbar_expect_tx(full(stage), 2 * kHalfTile / kLoadWarps);
        __syncwarp();
        const uint32_t dst = sa(stage) + (uint32_t)(kLoadRows * j * kBK * 2);
        if (loads) {
          if (whole && (kb + 1) * kBK <= g.k) {  // rows and columns inside x
            tc::tma_gather4_pair(dst, &map_a, kb * kBK, srow[0], srow[1], srow[2], srow[3], full_even(stage));
          } else {
#pragma unroll
            for (int i = 0; i < kLoadRows; ++i)
              tc::tma_load_2d_pair(dst + (uint32_t)(i * kBK * 2), &map_a, kb * kBK, srow[i], full_even(stage));
          }
        }
        if (++stage == kStagesP) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok && lane == 0) flag_error(g, 8);
  } else {
    // ---------------------------------------------------------------- epilogue (both CTAs)
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;  // column half (score) or quarter of the tile
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = cluster; tile < tiles; tile += clusters) {
      const int rb = tile / g.n_tiles, nt = tile - rb * g.n_tiles;
      if (!tc::mbar_wait_warp(tfull(acc), acc_phase)) {
        if (lane == 0) flag_error(g, 4);
        break;
      }
      tc::fence_after_sync();
      const int rb128 = 2 * rb + (int)rank;  // this CTA's 128-row block
      const long long row = (long long)rb128 * kBM + 32 * q + lane;
      const bool row_ok = row < g.m;
      const uint32_t taddr = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(acc * kBN);
      Acc sums{{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
      if (kMode == kModeScore)
        drain_tile<kMode>(g, taddr, half, nt, row, row_ok, sums);
      else
        drain_tile_store<epi_parts(kMode)>(g, &map_out, out_stage + (uint32_t)((warp - 2) * stage_out(kMode)), taddr,
                                           half, nt,
                         row - lane);
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive_cluster(tempty_even(acc));  // this warp is done with the accumulator
      if (kMode == kModeScore && rb128 * kBM < g.m) publish_rows(g, rb128, nt, half, q, row, row_ok, sums);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (kMode != kModeScore && lane == 0) tc::bulk_wait();  // this warp's output stores have completed
  }

  tc::fence_before_sync();
  tc::cluster_sync();  // neither CTA leaves while the other may still signal its barriers
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc_pair(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- host side
using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                 const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn() {
  static std::once_flag once;
  static EncodeTiled fn = nullptr;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiled>(p);
  });
  return fn;
}

// Row-major bf16 [rows, cols] read in boxes of box_rows x 64 columns with the
// 128-byte swizzle; out-of-range rows and columns read as zeros.
// A bf16 [rows, cols] row-major tensor in boxes of box_rows x box_cols
// (box_cols x 2 bytes = the swizzle span: 64 columns with the 128-byte
// swizzle for operands, 32 with the 64-byte swizzle for the output staging).
bool make_map(CUtensorMap *map, const void *base, long long rows, long long cols, int box_rows, int box_cols = kBK,
              CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  EncodeTiled fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<int> g_gemm_smem_set[64];

std::atomic<int> g_pair_smem_set[64];
std::atomic<int> g_pair_clusters[64][3];

template <int kMode>
cudaError_t launch_single(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mo, const GemmArgs &g,
                          cudaStream_t st, int dev) {
  const int bit = 1 << kMode;
  if (!(g_gemm_smem_set[dev & 63].load() & bit)) {
    cudaError_t err =
        cudaFuncSetAttribute(k_mlp_gemm<kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmem);
    if (err != cudaSuccess) return err;
    g_gemm_smem_set[dev & 63].fetch_or(bit);
  }
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const int grid = g.tiles < sms ? g.tiles : sms;
  k_mlp_gemm<kMode><<<grid, gemm_threads(kMode), kGemmSmem, st>>>(ma, mb, mo, g);
  return cudaGetLastError();
}

template <int kMode>
cudaError_t launch_pair(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mo, const GemmArgs &g,
                        cudaStream_t st, int dev) {
  const int bit = 1 << kMode;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(gemm_threads(kMode));
  cfg.dynamicSmemBytes = kGemmPSmem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (!(g_pair_smem_set[dev & 63].load() & bit)) {
    cudaError_t err = cudaFuncSetAttribute(k_mlp_gemm_pair<kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kGemmPSmem);
    if (err != cudaSuccess) return err;
    int clusters = 0;
    cfg.gridDim = dim3(2 * 64);
    err = cudaOccupancyMaxActiveClusters(&clusters, k_mlp_gemm_pair<kMode>, &cfg);
    if (err != cudaSuccess) return err;
    if (clusters <= 0) return cudaErrorInvalidConfiguration;
    g_pair_clusters[dev & 63][kMode].store(clusters);
    g_pair_smem_set[dev & 63].fetch_or(bit);
  }
  const int row_tiles = (g.m + 2 * kBM - 1) / (2 * kBM);
  const long long tiles = (long long)row_tiles * g.n_tiles;
  const int max_clusters = g_pair_clusters[dev & 63][kMode].load();
  const int clusters = tiles < max_clusters ? (int)tiles : max_clusters;
  cfg.gridDim = dim3(2 * clusters);
  return cudaLaunchKernelEx(&cfg, k_mlp_gemm_pair<kMode>, ma, mb, mo, g);
}

// Batches of more than one 128-row block run on SM pairs (2-SM MMA); a
// single row block on one SM.  The B operand's TMA box follows: 128 rows
// per CTA in a pair, the whole 256-row tile on one SM.
inline bool use_pair(int m) { return m > kBM; }
inline int b_box_rows(int m) { return use_pair(m) ? 128 : kBN; }

template <int kMode>
cudaError_t launch_gemm(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mo, const GemmArgs &g,
                        cudaStream_t st) {
  if (g.tiles == 0) return cudaSuccess;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  return use_pair(g.m) ? launch_pair<kMode>(ma, mb, mo, g, st, dev) : launch_single<kMode>(ma, mb, mo, g, st, dev);
}

bool misaligned16(const void *p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }

tr_status check_mlp(const tr_mlp *m) {
  if (!m || !m->x_pre || !m->w1 || !m->w2) return TR_ERR_ARG;
  if (m->t < 0 || m->d <= 0 || m->d_hidden <= 0) return TR_ERR_ARG;
  if (m->act != TR_ACT_GELU && m->act != TR_ACT_QUICK_GELU && m->act != TR_ACT_NONE) return TR_ERR_ARG;
  if (m->d % 16 != 0 || m->d_hidden % 16 != 0) return TR_ERR_ALIGN;
  if (m->d > TR_MAX_D || m->d_hidden > TR_MLP_MAX_HIDDEN) return TR_ERR_UNSUPPORTED;
  const long long rblocks = ((long long)m->t + kBM - 1) / kBM;  // tile counts stay in int
  if (rblocks * ((m->d_hidden + kBN - 1) / kBN) > INT_MAX) return TR_ERR_UNSUPPORTED;
  if (misaligned16(m->x_pre) || misaligned16(m->resid) || misaligned16(m->w1) || misaligned16(m->w2) ||
      misaligned16(m->b1) || misaligned16(m->b2))
    return TR_ERR_ALIGN;
  return TR_OK;
}

struct MlpWs {
  size_t part, arrivals, total;
};
MlpWs mlp_ws(const tr_mlp *m) {
  const long long rblocks = ((long long)m->t + kBM - 1) / kBM;
  const long long n_tiles = (m->d + kBN - 1) / kBN;
  MlpWs w;
  w.part = 0;
  w.arrivals = align_up((size_t)rblocks * n_tiles * 2 * 4 * kPartWords * 32 * sizeof(float), 256);
  w.total = align_up(w.arrivals + (size_t)rblocks * 4 * sizeof(int), 256);
  return w;
}

// out = act(a W^T + bias) for dense bf16 rows a [rows, k] and W [n, k]: the
// hidden-mode GEMM (bias + activation epilogue, TMA stores), arguments
// checked by the caller.
tr_status dense_act_gemm(const void *a, int rows, int k, const void *w, const float *bias, int n, int act, void *out,
                         int32_t *d_error, cudaStream_t st) {
  if (rows == 0) return TR_OK;
  GemmArgs g{};
  g.m = rows;
  g.n = n;
  g.k = k;
  g.n_tiles = (g.n + kBN - 1) / kBN;
  g.tiles = ((g.m + kBM - 1) / kBM) * g.n_tiles;
  g.kblocks = (g.k + kBK - 1) / kBK;
  g.bias = bias;
  g.act = act;
  g.out = static_cast<uint16_t *>(out);
  g.err = d_error;
  CUtensorMap ma, mb, mo;
  if (!make_map(&ma, a, rows, k, kBM) || !make_map(&mb, w, n, k, b_box_rows(g.m)) ||
      !make_map(&mo, out, rows, n, 32, 128 / epi_parts(kModeHidden),
                epi_parts(kModeHidden) == 2 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
    return TR_ERR_CUDA;
  return launch_gemm<kModeHidden>(ma, mb, mo, g, st) == cudaSuccess ? TR_OK : TR_ERR_CUDA;
}

}  // namespace
}  // namespace tr

using namespace tr;

extern "C" {

tr_status tr_mlp_hidden(const tr_mlp *m, void *h, int32_t *d_error, void *stream) {
  tr_status rc = check_mlp(m);
  if (rc != TR_OK) return rc;
  if (!h) return TR_ERR_ARG;
  if (misaligned16(h)) return TR_ERR_ALIGN;
  return dense_act_gemm(m->x_pre, m->t, m->d, m->w1, m->b1, m->d_hidden, m->act, h, d_error,
                        static_cast<cudaStream_t>(stream));
}

tr_status tr_project(const void *y, int32_t rows, int32_t d, const void *w, const float *bias, int32_t d_out,
                     int32_t act, void *z, int32_t *d_error, void *stream) {
  if (!y || !w || !z || rows < 0 || d <= 0 || d_out <= 0) return TR_ERR_ARG;
  if (act != TR_ACT_GELU && act != TR_ACT_QUICK_GELU && act != TR_ACT_NONE) return TR_ERR_ARG;
  if (d % 16 != 0 || d_out % 16 != 0) return TR_ERR_ALIGN;
  if (d > TR_MAX_D || d_out > TR_MLP_MAX_HIDDEN) return TR_ERR_UNSUPPORTED;
  if (((long long)rows + kBM - 1) / kBM * ((d_out + kBN - 1) / kBN) > INT_MAX) return TR_ERR_UNSUPPORTED;
  if (misaligned16(y) || misaligned16(w) || misaligned16(bias) || misaligned16(z)) return TR_ERR_ALIGN;
  return dense_act_gemm(y, rows, d, w, bias, d_out, act, z, d_error, static_cast<cudaStream_t>(stream));
}

size_t tr_mlp_workspace_bytes(const tr_mlp *m) {
  if (check_mlp(m) != TR_OK) return 0;
  return mlp_ws(m).total;
}

tr_status tr_mlp_score(const tr_mlp *m, const void *h, void *x_post, void *x, float *stats, float *h2, float *s,
                       void *ws, size_t ws_bytes, int32_t *d_error, void *stream) {
  tr_status rc = check_mlp(m);
  if (rc != TR_OK) return rc;
  if (!h || !x_post || !x || !stats) return TR_ERR_ARG;
  if (misaligned16(h) || misaligned16(x_post) || misaligned16(x) || misaligned16(stats) ||
      (reinterpret_cast<uintptr_t>(h2) & 3u) || (reinterpret_cast<uintptr_t>(s) & 3u))
    return TR_ERR_ALIGN;
  const MlpWs w = mlp_ws(m);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < w.total) return TR_ERR_WORKSPACE;
  if (m->t == 0) return TR_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char *wsb = static_cast<char *>(ws);
  if (cudaMemsetAsync(wsb + w.arrivals, 0, w.total - w.arrivals, st) != cudaSuccess) return TR_ERR_CUDA;
  GemmArgs g{};
  g.m = m->t;
  g.n = m->d;
  g.k = m->d_hidden;
  g.n_tiles = (g.n + kBN - 1) / kBN;
  g.tiles = ((g.m + kBM - 1) / kBM) * g.n_tiles;
  g.kblocks = (g.k + kBK - 1) / kBK;
  g.bias = m->b2;
  g.out = static_cast<uint16_t *>(x_post);
  g.x_pre = static_cast<const uint16_t *>(m->x_pre);
  g.resid = static_cast<const uint16_t *>(m->resid);
  g.x = static_cast<uint16_t *>(x);
  g.part = reinterpret_cast<float *>(wsb + w.part);
  g.arrivals = reinterpret_cast<int *>(wsb + w.arrivals);
  g.stats = reinterpret_cast<float4 *>(stats);
  g.h2 = h2;
  g.s = s;
  g.err = d_error;
  CUtensorMap ma, mb;
  if (!make_map(&ma, h, m->t, m->d_hidden, kBM) || !make_map(&mb, m->w2, m->d, m->d_hidden, b_box_rows(g.m)))
    return TR_ERR_CUDA;
  return launch_gemm<kModeScore>(ma, mb, mb, g, st) == cudaSuccess ? TR_OK : TR_ERR_CUDA;  // no output map
}

tr_status tr_project_kept(const tr_tokens *in, const int32_t *d_cu_k, const int32_t *idx, int32_t total_k,
                          const void *w, const float *bias, int32_t d_out, int32_t act, void *z, int32_t *d_error,
                          void *stream) {
  if (!in || !in->x || !w || !z) return TR_ERR_ARG;
  if (in->dtype != TR_BF16) return TR_ERR_DTYPE;
  if (in->d <= 0 || d_out <= 0 || in->batch < 0) return TR_ERR_ARG;
  if (act != TR_ACT_GELU && act != TR_ACT_QUICK_GELU && act != TR_ACT_NONE) return TR_ERR_ARG;
  if (in->d % 16 != 0 || d_out % 16 != 0) return TR_ERR_ALIGN;
  if (in->d > TR_MAX_D || d_out > TR_MLP_MAX_HIDDEN) return TR_ERR_UNSUPPORTED;
  if (misaligned16(in->x) || misaligned16(w) || misaligned16(bias) || misaligned16(z)) return TR_ERR_ALIGN;
  long long total_rows;
  if (in->cu_seqlens) {
    if (in->total < 0) return TR_ERR_ARG;
    total_rows = in->total;
  } else {
    if (in->n < 0) return TR_ERR_ARG;
    total_rows = (long long)in->batch * in->n;
  }
  if (total_k < 0 || total_k > total_rows) return TR_ERR_BUDGET;
  if (total_rows > INT_MAX) return TR_ERR_UNSUPPORTED;  // TMA row coordinates are 32-bit
  if (total_k == 0) return TR_OK;
  if (in->batch == 0 || !d_cu_k || !idx) return TR_ERR_ARG;
  const long long rblocks = ((long long)total_k + kBM - 1) / kBM;
  if (rblocks * ((d_out + kBN - 1) / kBN) > INT_MAX) return TR_ERR_UNSUPPORTED;
  GemmArgs g{};
  g.m = total_k;
  g.n = d_out;
  g.k = in->d;
  g.n_tiles = (g.n + kBN - 1) / kBN;
  g.tiles = (int)rblocks * g.n_tiles;
  g.kblocks = (g.k + kBK - 1) / kBK;
  g.bias = bias;
  g.act = act;
  g.out = static_cast<uint16_t *>(z);
  g.err = d_error;
  g.gx = static_cast<const uint16_t *>(in->x);
  g.total_rows = total_rows;
  g.batch = in->batch;
  g.n_uniform = in->cu_seqlens ? 0 : in->n;
  g.cu_seqlens = in->cu_seqlens;
  g.cu_k = d_cu_k;
  g.idx = idx;
  // A: x, one row per box (the loaders gather rows by kept index)
  CUtensorMap ma, mb, mo;
  if (!make_map(&ma, in->x, total_rows, in->d, 1) || !make_map(&mb, w, d_out, in->d, b_box_rows(g.m)) ||
      !make_map(&mo, z, total_k, d_out, 32, 128 / epi_parts(kModeProject),
                epi_parts(kModeProject) == 2 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
    return TR_ERR_CUDA;
  return launch_gemm<kModeProject>(ma, mb, mo, g, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TR_OK
                                                                                                     : TR_ERR_CUDA;
}

}  // extern "C"
