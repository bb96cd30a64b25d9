// Gather of the kept tokens: y[r] = x[row_off(b) + idx[r]] for the image b
// that owns output row r (cu_k[b] <= r < cu_k[b+1]), a bit copy of d * elem
// bytes per row (Eq. 7: X* is made of the original token vectors).  One warp
// per output row, 16-byte loads that skip L1 and streaming stores.
#include "tr_internal.cuh"

namespace tr {
namespace {

__device__ __forceinline__ uint4 ld_nc(const uint4 *p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}
__device__ __forceinline__ void st_cs(uint4 *p, const uint4 &v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

__global__ void __launch_bounds__(kGatherWarps * 32)
    k_gather(const uint4 *__restrict__ x, long long total_rows, int batch, int n_uniform,
             const int32_t *__restrict__ cu_seqlens, const int32_t *__restrict__ cu_k,
             const int32_t *__restrict__ idx, int total_k, int nchunks, uint4 *__restrict__ y) {
  pdl_wait();  // idx comes from the kernel before this one
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * kGatherWarps + (threadIdx.x >> 5);
  if (row >= total_k) return;
  // image b: the last b with cu_k[b] <= row (skipping images with K_b = 0)
  int lo = 0, hi = batch;  // invariant: cu_k[lo] <= row < cu_k[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(cu_k + mid) <= row) lo = mid; else hi = mid;
  }
  const long long first = cu_seqlens ? (long long)__ldg(cu_seqlens + lo) : (long long)lo * n_uniform;
  const long long n_b = cu_seqlens ? (long long)__ldg(cu_seqlens + lo + 1) - first : (long long)n_uniform;
  const int local = __ldcg(idx + row);  // through L2: idx may come from the kernel before
  const long long g = first + local;
  uint4 *dst = y + (long long)row * nchunks;
  // an index outside its own image's tokens (or an image outside x) writes
  // zeros: never a row of another image, never an address outside x
  if (local < 0 || local >= n_b || first < 0 || g >= total_rows) {
    for (int c = lane; c < nchunks; c += 32) st_cs(dst + c, make_uint4(0u, 0u, 0u, 0u));
    return;
  }
  const uint4 *src = x + (long long)g * nchunks;
  constexpr int kU = 4;  // loads in flight per lane (8, and 2- or 4-warp CTAs, measured no faster)
  int c = lane;
  for (; c + 32 * (kU - 1) < nchunks; c += 32 * kU) {
    uint4 v[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) v[u] = ld_nc(src + c + 32 * u);
#pragma unroll
    for (int u = 0; u < kU; ++u) st_cs(dst + c + 32 * u, v[u]);
  }
  for (; c < nchunks; c += 32) st_cs(dst + c, ld_nc(src + c));
}

}  // namespace

cudaError_t launch_gather(const void *x, long long total_rows, int dtype, int d, int batch, int n_uniform,
                          const int32_t *cu_seqlens, const int32_t *cu_k, const int32_t *idx, int total_k, void *y,
                          cudaStream_t st, bool pdl) {
  if (total_k == 0) return cudaSuccess;
  const int nchunks = d * elem_bytes(dtype) / 16;
  const int grid = (total_k + kGatherWarps - 1) / kGatherWarps;
  return launch_kernel(k_gather, dim3(grid), dim3(kGatherWarps * 32), 0, st, pdl, static_cast<const uint4 *>(x),
                       total_rows, batch, n_uniform, cu_seqlens, cu_k, idx, total_k, nchunks,
                       static_cast<uint4 *>(y));
}

}  // namespace tr
