// The selection kernel: one CTA per image runs select_image (Algorithm 1,
// see tr_select_dev.cuh) on statistics left by the scoring kernel.
#include "tr_select_dev.cuh"

namespace tr {
namespace {

__global__ void __launch_bounds__(kSelectThreads, 1) k_select(const SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  select_image(a, blockIdx.x, smem);
}

int g_smem_set[64];  // per device: dynamic shared memory limit already raised

}  // namespace

size_t select_smem_bytes(int max_n) {
  const size_t cap = (size_t)row_capacity(max_n > 0 ? max_n : 1);
  return cap * (sizeof(uint32_t) + 2 * sizeof(uint16_t) + sizeof(uint8_t)) + kWarps * 256 * sizeof(uint32_t);
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
    cudaFuncAttributes fa;
    err = cudaFuncGetAttributes(&fa, k_select);
    if (err != cudaSuccess) return err;
    err = cudaFuncSetAttribute(k_select, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
    if (err != cudaSuccess) return err;
    g_smem_set[dev & 63] = 1;
  }
  k_select<<<a.batch, kSelectThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace tr
