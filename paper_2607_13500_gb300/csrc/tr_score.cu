// Scoring pass (Eq. 3-4 and Eq. 6): one warp per row over a grid of resident
// CTAs; the row arithmetic is in tr_score_dev.cuh.
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
  const int row_bytes = d * elem_bytes(dtype);
  const unsigned char *bx = static_cast<const unsigned char *>(x);
  const unsigned char *bp = static_cast<const unsigned char *>(x_pre ? x_pre : x);
  const unsigned char *bq = static_cast<const unsigned char *>(x_post);
  float4 *ps = reinterpret_cast<float4 *>(stats);
  const long long need = (total + kScoreWarps - 1) / kScoreWarps;
  const long long cap = (long long)info.sms * info.blocks_per_sm[which];
  const int grid = (int)(need < cap ? need : cap);
  const int nchunks = row_bytes / 16;
  const uint4 *px = reinterpret_cast<const uint4 *>(bx);
  const uint4 *pp = reinterpret_cast<const uint4 *>(bp);
  const uint4 *pq = reinterpret_cast<const uint4 *>(bq);
  if (which)
    k_score<true><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  else
    k_score<false><<<grid, kScoreWarps * 32, 0, st>>>(px, pp, pq, nchunks, total, ps, h2, s);
  return cudaGetLastError();
}

}  // namespace tr
