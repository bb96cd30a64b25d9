// Scoring pass (Eq. 3-4 and Eq. 6): one warp per row, one CTA per
// kScoreWarps rows; the row arithmetic is in tr_score_dev.cuh.
#include <climits>

#include "tr_score_dev.cuh"

namespace tr {
namespace {

template <int kDt>
__global__ void __launch_bounds__(kScoreWarps * 32)
    k_score(const uint4 *__restrict__ x, const uint4 *__restrict__ xp, const uint4 *__restrict__ xq, int nchunks,
            long long total, float4 *__restrict__ stats, float *__restrict__ h2, float *__restrict__ s_out) {
  pdl_trigger();  // a dependent selection may be scheduled once every CTA runs
  const int lane = threadIdx.x & 31;
  const long long stride = (long long)gridDim.x * kScoreWarps;
  for (long long row = (long long)blockIdx.x * kScoreWarps + (threadIdx.x >> 5); row < total; row += stride)
    score_row<kDt>(x, xp, xq, nchunks, row, stats, h2, s_out, lane);
}

}  // namespace

cudaError_t launch_score(const void *x, const void *x_pre, const void *x_post, int dtype, int d, long long total,
                         float *stats, float *h2, float *s, cudaStream_t st) {
  if (total == 0) return cudaSuccess;
  const int row_bytes = d * elem_bytes(dtype);
  const unsigned char *bx = static_cast<const unsigned char *>(x);
  const unsigned char *bp = static_cast<const unsigned char *>(x_pre ? x_pre : x);
  const unsigned char *bq = static_cast<const unsigned char *>(x_post);
  float4 *ps = reinterpret_cast<float4 *>(stats);
  // One row per warp and no more, in small CTAs: CTAs retire as they
  // finish, so kernels on other streams (the selection of an earlier batch)
  // can take SMs while this one still runs, and an SM's slots refill row by
  // row.  (Measured on GB300: 2-warp CTAs beat 1-, 4-, 8- and 16-warp ones
  // and 2 or 4 rows per warp; a persistent grid is no faster alone and would
  // hold every SM to the end.)
  const long long need = (total + kScoreWarps - 1) / kScoreWarps;
  const int grid = (int)(need < INT_MAX ? need : INT_MAX);
  const int nchunks = row_bytes / 16;
  const uint4 *px = reinterpret_cast<const uint4 *>(bx);
  const uint4 *pp = reinterpret_cast<const uint4 *>(bp);
  const uint4 *pq = reinterpret_cast<const uint4 *>(bq);
  if (dtype == TR_BF16)
    k_score<TR_BF16><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  else if (dtype == TR_F16)
    k_score<TR_F16><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  else
    k_score<TR_F32><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  return cudaGetLastError();
}

}  // namespace tr
