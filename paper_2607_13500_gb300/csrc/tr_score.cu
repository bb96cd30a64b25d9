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
// than fp32.  The epilogue rounds the sums to fp32 and derives the fp32
// selection keys, all without fp64 (GB300's fp64 rate would stall the warp).
#include "tr_score_dev.cuh"

namespace tr {
namespace {

template <bool kBf16>
__global__ void __launch_bounds__(kScoreWarps * 32)
    k_score(const uint4 *__restrict__ x, const uint4 *__restrict__ xp, const uint4 *__restrict__ xq, int nchunks,
            long long total, float4 *__restrict__ stats, float *__restrict__ h2, float *__restrict__ s_out) {
  const int lane = threadIdx.x & 31;
  const long long stride = (long long)gridDim.x * kScoreWarps;
  for (long long row = (long long)blockIdx.x * kScoreWarps + (threadIdx.x >> 5); row < total; row += stride)
    score_row<kBf16>(x, xp, xq, nchunks, row, stats, h2, s_out, lane);
}

struct DevInfo {
  int sms = 0;
  int blocks_per_sm[2] = {0, 0};
};

DevInfo &dev_info(int dev) {
  static DevInfo info[64];
  return info[dev & 63];
}

}  // namespace

cudaError_t launch_score(const void *x, const void *x_pre, const void *x_post, int dtype, int d, long long total,
                         float *stats, float *h2, float *s, cudaStream_t st) {
  if (total == 0) return cudaSuccess;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  DevInfo &info = dev_info(dev);
  const int which = dtype == TR_BF16 ? 1 : 0;
  if (info.blocks_per_sm[which] == 0) {
    // Benign race: concurrent first calls compute the same numbers.
    int sms = 0, bps = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    err = which ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, k_score<true>, kScoreWarps * 32, 0)
                : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bps, k_score<false>, kScoreWarps * 32, 0);
    if (err != cudaSuccess) return err;
    info.sms = sms;
    info.blocks_per_sm[which] = bps > 0 ? bps : 1;
  }
  const long long need = (total + kScoreWarps - 1) / kScoreWarps;
  const long long cap = (long long)info.sms * info.blocks_per_sm[which];
  const int grid = (int)(need < cap ? need : cap);
  const int nchunks = d * elem_bytes(dtype) / 16;
  const uint4 *px = static_cast<const uint4 *>(x);
  const uint4 *pp = static_cast<const uint4 *>(x_pre ? x_pre : x);
  const uint4 *pq = static_cast<const uint4 *>(x_post);
  float4 *ps = reinterpret_cast<float4 *>(stats);
  if (which)
    k_score<true><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  else
    k_score<false><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  return cudaGetLastError();
}

}  // namespace tr
