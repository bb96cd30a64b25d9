// tr_reduce_noalloc: the whole reduction for callers that cannot allocate
// device memory themselves.
//
// Some callers have no way to obtain a device workspace: code that runs
// inside a host framework whose allocator it cannot reach, plugin or
// callback code that is forbidden to call cudaMalloc on its hot path, or
// real-time loops that must not allocate at all once they are running.  For
// them this entry point takes its scratch (the per-row statistics and the
// exact-sum records of the selection) from a file-scope device array instead
// of a caller-provided workspace.
//
// The array is TR_NOALLOC_SCRATCH_BYTES bytes (enough for
// TR_NOALLOC_MAX_ROWS token rows) and exists on every GPU that loads this
// library, for as long as the library stays loaded.  All calls share it, so
// calls whose work overlaps on the GPU (different streams, or different
// host threads on one device) race on it and must be serialised by the
// caller.  Nothing in it has to start at zero: the scoring pass overwrites
// every statistics row it uses, and the selection writes an exact record
// before it reads one.
#include <mutex>

#include "tr_internal.cuh"

namespace {

// The device address of the array is looked up once per device, with that
// device current, on the first call made there.
__device__ __align__(256) unsigned char g_scratch[TR_NOALLOC_SCRATCH_BYTES];

std::mutex g_mu;
void *g_scratch_ptr[64];

tr_status scratch_address(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return TR_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) return TR_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return TR_OK;
}

}  // namespace

extern "C" tr_status tr_reduce_noalloc(const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1,
                                       const int32_t *d_cu_k, int32_t total_k, void *y, int32_t *idx, float *h2,
                                       float *s, int32_t *d_status, void *stream) {
  if (!in) return TR_ERR_ARG;
  const long long rows = in->cu_seqlens ? (long long)in->total : (long long)in->batch * in->n;
  if (rows > TR_NOALLOC_MAX_ROWS) return TR_ERR_UNSUPPORTED;
  const size_t need = tr_workspace_bytes(in);
  if (need > (size_t)TR_NOALLOC_SCRATCH_BYTES) return TR_ERR_UNSUPPORTED;
  void *scratch = nullptr;
  const tr_status rc = scratch_address(&scratch);
  if (rc != TR_OK) return rc;
  return tr_reduce(in, d_k, d_k1, d_cu_k, total_k, y, idx, h2, s, scratch, (size_t)TR_NOALLOC_SCRATCH_BYTES,
                   d_status, stream);
}
