// The selection kernels: a CTA runs select_image (Algorithm 1, see
// tr_select_dev.cuh) on statistics left by the scoring kernel, one image at
// a time (k_select: one image per CTA, or several in turn when the launch
// caps the grid, as the pipeline does).
//
// k_select_gather (tr_reduce on uniform batches) also copies the kept rows.
// With fewer images than SMs it runs R replica CTAs per image: each makes
// the same deterministic selection (only replica 0 writes idx and the status
// words) and copies its 1/R share of the image's kept rows, so the copies of
// one image overlap the selections of the others on SMs that would be idle.
#include <atomic>

#include "tr_select_dev.cuh"

namespace tr {
namespace {

// CTA c selects images c, c + gridDim.x, ... (one image per CTA unless the
// launch caps the grid below the batch).
__global__ void __launch_bounds__(kSelectThreads, 1) k_select(const SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  pdl_trigger();
  pdl_wait();  // the statistics come from the kernel before this one
  for (int b = blockIdx.x; b < a.batch; b += gridDim.x) select_image(a, b, smem);
}

__device__ __forceinline__ uint4 ld_nc16(const uint4 *p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

// Replica r of `replicas` copies its share of image b's kept rows, whose
// local indices select_image left in this CTA's shared memory.
__device__ __forceinline__ void copy_kept(const SelectArgs &a, const int b, const int r, const int replicas,
                                          const int nchunks, uint4 *__restrict__ y, unsigned char *smem) {
  long long off;
  int n;
  if (a.cu_seqlens) {
    off = a.cu_seqlens[b];
    n = a.cu_seqlens[b + 1] - a.cu_seqlens[b];
  } else {
    off = (long long)b * a.n_uniform;
    n = a.n_uniform;
  }
  const int k = a.k[b], k1 = a.k1[b], ko = a.cu_k[b];
  if (n <= 0 || n > a.max_n || off < 0 || off + n > a.total_rows || k < 0 || k > n || k1 < 0 || k1 > k)
    return;  // counted by select_image
  // this replica's share of the image's kept rows
  const uint16_t *kept = kept_rows(a, smem);
  const int j0 = (int)((long long)r * k / replicas), j1 = (int)((long long)(r + 1) * k / replicas);
  const uint4 *x = static_cast<const uint4 *>(a.x);
  // one warp per row, eight 16-byte loads in flight per lane, streaming stores
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kU = 8;
  for (int j = j0 + warp; j < j1; j += kWarps) {
    const uint4 *src = x + (off + kept[j]) * nchunks;
    uint4 *dst = y + (long long)(ko + j) * nchunks;
    for (int c0 = lane; c0 < nchunks; c0 += 32 * kU) {
      uint4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int c = c0 + 32 * u;
        if (c < nchunks) v[u] = ld_nc16(src + c);
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int c = c0 + 32 * u;
        if (c < nchunks) __stcs(dst + c, v[u]);
      }
    }
  }
}

__global__ void __launch_bounds__(kSelectThreads, 1)
    k_select_gather(const SelectArgs a, const int replicas, const int nchunks, uint4 *__restrict__ y) {
  extern __shared__ __align__(16) unsigned char smem[];
  pdl_wait();  // the statistics come from the kernel before this one
  const int b = blockIdx.x / replicas, r = blockIdx.x % replicas;
  select_image(a, b, smem, r == 0);
  copy_kept(a, b, r, replicas, nchunks, y, smem);
}

// Per device (index & 63): dynamic shared memory limit already raised (bit 0
// k_select, bit 1 k_select_gather), and the SM count.  Atomic so that first
// calls from several host threads are well defined (raising the limit twice
// is harmless).
std::atomic<int> g_smem_set[64];
std::atomic<int> g_sms[64];

}  // namespace

size_t select_smem_bytes(int max_n) {
  const size_t cap = (size_t)row_capacity(max_n > 0 ? max_n : 1);
  return cap * (sizeof(uint32_t) + 3 * sizeof(uint16_t) + sizeof(uint8_t)) + kWarps * 256 * sizeof(uint32_t);
}

template <typename K>
cudaError_t raise_smem_limit(K kernel, int dev) {
  int optin = 0;
  cudaError_t err = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (err != cudaSuccess) return err;
  cudaFuncAttributes fa;
  err = cudaFuncGetAttributes(&fa, kernel);
  if (err != cudaSuccess) return err;
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
}

cudaError_t launch_select(const SelectArgs &a, cudaStream_t st, int max_ctas, bool pdl) {
  if (a.batch == 0) return cudaSuccess;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const size_t smem = select_smem_bytes(a.max_n);
  if (!(g_smem_set[dev & 63].load() & 1)) {
    if ((err = raise_smem_limit(k_select, dev)) != cudaSuccess) return err;
    g_smem_set[dev & 63].fetch_or(1);
  }
  const int grid = max_ctas > 0 && max_ctas < a.batch ? max_ctas : a.batch;
  return launch_kernel(k_select, dim3(grid), dim3(kSelectThreads), smem, st, pdl, a);
}

int sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (!g_sms[dev & 63].load()) {
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    g_sms[dev & 63].store(sms);
  }
  return g_sms[dev & 63].load();
}

cudaError_t launch_select_gather(const SelectArgs &a, void *y, cudaStream_t st, bool pdl) {
  if (a.batch == 0) return cudaSuccess;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (!(g_smem_set[dev & 63].load() & 2)) {
    if ((err = raise_smem_limit(k_select_gather, dev)) != cudaSuccess) return err;
    g_smem_set[dev & 63].fetch_or(2);
  }
  const int sms = sm_count();
  if (sms <= 0) return cudaErrorInvalidDevice;
  const size_t smem = select_smem_bytes(a.max_n);
  const int nchunks = a.d * elem_bytes(a.dtype) / 16;
  const int replicas = max(1, min(16, sms / a.batch));
  return launch_kernel(k_select_gather, dim3(a.batch * replicas), dim3(kSelectThreads), smem, st, pdl, a, replicas,
                       nchunks, static_cast<uint4 *>(y));
}

}  // namespace tr
