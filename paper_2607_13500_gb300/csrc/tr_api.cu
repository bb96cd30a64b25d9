// Host side of the C ABI declared in include/tr.h: argument checks, budgets,
// workspace carving and launches (tr_reduce: score, then select + gather).
#include <algorithm>
#include <climits>

#include <new>

#include "tr_internal.cuh"

using namespace tr;

namespace {

bool misaligned(const void *p, uintptr_t a) { return p && (reinterpret_cast<uintptr_t>(p) % a) != 0; }

struct Shape {
  long long total;
  int max_n;
};

tr_status check_tokens(const tr_tokens *in, Shape *sh) {
  if (!in || !in->x || !in->x_post) return TR_ERR_ARG;
  if (in->dtype != TR_F32 && in->dtype != TR_BF16 && in->dtype != TR_F16) return TR_ERR_DTYPE;
  if (in->flags & ~TR_STRIDE_INTERVAL) return TR_ERR_ARG;
  if (in->d <= 0 || in->batch < 0) return TR_ERR_ARG;
  if (in->d > TR_MAX_D) return TR_ERR_UNSUPPORTED;
  if ((in->d * elem_bytes(in->dtype)) % 16 != 0) return TR_ERR_ALIGN;
  if (misaligned(in->x, 16) || misaligned(in->x_pre, 16) || misaligned(in->x_post, 16)) return TR_ERR_ALIGN;
  if (in->cu_seqlens) {
    if (in->total < 0 || in->max_n < 0) return TR_ERR_ARG;
    sh->total = in->total;
    sh->max_n = in->max_n;
  } else {
    if (in->n < 0) return TR_ERR_ARG;
    sh->total = (long long)in->batch * in->n;
    sh->max_n = in->n;
  }
  if (sh->max_n > TR_MAX_N) return TR_ERR_UNSUPPORTED;
  if (sh->total > INT_MAX) return TR_ERR_UNSUPPORTED;  // kept rows are int32
  return TR_OK;
}

tr_status check_ws(const Shape &sh, const void *ws, size_t ws_bytes) {
  if (!ws || misaligned(ws, 256)) return TR_ERR_WORKSPACE;
  if (ws_bytes < ws_layout(sh.total).total) return TR_ERR_WORKSPACE;
  return TR_OK;
}

SelectArgs select_args(const tr_tokens *in, const Shape &sh, const float *stats, const int32_t *d_k,
                       const int32_t *d_k1, const int32_t *d_cu_k, int32_t *idx, uint8_t *role,
                       float *h2, float *s, void *ws, int32_t *d_status) {
  SelectArgs a;
  a.x = in->x;
  a.x_pre = in->x_pre;
  a.x_post = in->x_post;
  a.dtype = in->dtype;
  a.d = in->d;
  a.batch = in->batch;
  a.n_uniform = in->cu_seqlens ? 0 : in->n;
  a.cu_seqlens = in->cu_seqlens;
  a.stats = stats;
  a.k = d_k;
  a.k1 = d_k1;
  a.cu_k = d_cu_k;
  a.idx = idx;
  a.role = role;
  a.h2 = h2;
  a.s = s;
  a.exact = reinterpret_cast<ExactRec *>(static_cast<char *>(ws) + ws_layout(sh.total).exact);
  a.status = d_status;
  a.bounds = certification_bounds(in->d, in->dtype);
  a.max_n = sh.max_n;
  a.total_rows = sh.total;
  a.stride_interval = (in->flags & TR_STRIDE_INTERVAL) != 0;
  return a;
}

tr_status select_capped(const tr_tokens *in, const float *stats, const int32_t *d_k, const int32_t *d_k1,
                        const int32_t *d_cu_k, int32_t *idx, uint8_t *role, float *h2, float *s, void *ws,
                        size_t ws_bytes, int32_t *d_status, void *stream, int max_ctas, bool pdl) {
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (in->batch > 0 && (!stats || !d_k || !d_k1 || !d_cu_k || !idx)) return TR_ERR_ARG;
  if (misaligned(stats, 16)) return TR_ERR_ALIGN;
  if ((rc = check_ws(sh, ws, ws_bytes)) != TR_OK) return rc;
  SelectArgs a = select_args(in, sh, stats, d_k, d_k1, d_cu_k, idx, role, h2, s, ws, d_status);
  cudaError_t err = launch_select(a, static_cast<cudaStream_t>(stream), max_ctas, pdl);
  return err == cudaSuccess ? TR_OK : TR_ERR_CUDA;
}

tr_status gather_impl(const tr_tokens *in, const int32_t *d_cu_k, const int32_t *idx, int32_t total_k, void *y,
                      void *stream, bool pdl) {
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (total_k < 0 || total_k > sh.total) return TR_ERR_BUDGET;
  if (total_k > 0 && (!d_cu_k || !idx || !y || in->batch == 0)) return TR_ERR_ARG;
  if (misaligned(y, 16)) return TR_ERR_ALIGN;
  cudaError_t err = launch_gather(in->x, sh.total, in->dtype, in->d, in->batch, in->cu_seqlens ? 0 : in->n,
                                  in->cu_seqlens, d_cu_k, idx, total_k, y, static_cast<cudaStream_t>(stream), pdl);
  return err == cudaSuccess ? TR_OK : TR_ERR_CUDA;
}

}  // namespace

extern "C" {

const char *tr_status_string(int32_t status) {
  switch (status) {
    case TR_OK: return "ok";
    case TR_ERR_ARG: return "invalid argument";
    case TR_ERR_BUDGET: return "invalid budget";
    case TR_ERR_DTYPE: return "unsupported dtype";
    case TR_ERR_ALIGN: return "misaligned row or pointer (rows must be a multiple of 16 bytes)";
    case TR_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case TR_ERR_CUDA: return "CUDA launch failed";
    case TR_ERR_UNSUPPORTED: return "size above the supported maximum";
    default: return "unknown status";
  }
}

const char *tr_version(void) { return "libtr 0.1 (sm_103a)"; }

tr_status tr_budgets(int32_t batch, const int32_t *h_seqlens, int32_t k, int32_t r_num, int32_t r_den,
                     int32_t lam_num, int32_t lam_den, int32_t *h_k, int32_t *h_k1, int32_t *h_cu_k) {
  if (batch < 0 || !h_cu_k || (batch > 0 && (!h_seqlens || !h_k || !h_k1))) return TR_ERR_ARG;
  if (lam_den <= 0 || lam_num < 0 || lam_num > lam_den) return TR_ERR_BUDGET;
  if (k <= 0 && (r_den <= 0 || r_num <= 0 || r_num > r_den)) return TR_ERR_BUDGET;
  long long cum = 0;
  h_cu_k[0] = 0;
  for (int b = 0; b < batch; ++b) {
    const long long n = h_seqlens[b];
    if (n < 0) return TR_ERR_ARG;
    long long kb;
    if (k > 0)
      kb = k;
    else
      kb = n == 0 ? 0 : (n * r_num / r_den > 0 ? n * r_num / r_den : 1);
    if (kb > n) return TR_ERR_BUDGET;
    cum += kb;
    if (cum > INT_MAX) return TR_ERR_UNSUPPORTED;
    h_k[b] = (int32_t)kb;
    h_k1[b] = (int32_t)(kb * lam_num / lam_den);
    h_cu_k[b + 1] = (int32_t)cum;
  }
  return TR_OK;
}

size_t tr_workspace_bytes(const tr_tokens *in) {
  Shape sh;
  if (check_tokens(in, &sh) != TR_OK) return 0;
  return ws_layout(sh.total).total;
}

tr_status tr_score(const tr_tokens *in, float *stats, float *h2, float *s, void *stream) {
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (!stats) return TR_ERR_ARG;
  if (misaligned(stats, 16) || misaligned(h2, 4) || misaligned(s, 4)) return TR_ERR_ALIGN;
  cudaError_t err = launch_score(in->x, in->x_pre, in->x_post, in->dtype, in->d, sh.total, stats, h2, s,
                                 static_cast<cudaStream_t>(stream));
  return err == cudaSuccess ? TR_OK : TR_ERR_CUDA;
}

tr_status tr_select(const tr_tokens *in, const float *stats, const int32_t *d_k, const int32_t *d_k1,
                    const int32_t *d_cu_k, int32_t *idx, uint8_t *role, float *h2, float *s, void *ws,
                    size_t ws_bytes, int32_t *d_status, void *stream) {
  return select_capped(in, stats, d_k, d_k1, d_cu_k, idx, role, h2, s, ws, ws_bytes, d_status, stream, 0, true);
}

tr_status tr_select_gather(const tr_tokens *in, const float *stats, const int32_t *d_k, const int32_t *d_k1,
                           const int32_t *d_cu_k, int32_t total_k, void *y, int32_t *idx, float *h2, float *s,
                           void *ws, size_t ws_bytes, int32_t *d_status, void *stream) {
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (total_k < 0 || total_k > sh.total) return TR_ERR_BUDGET;
  if (in->batch > 0 && (!stats || !d_k || !d_k1 || !d_cu_k || !idx || (total_k > 0 && !y))) return TR_ERR_ARG;
  if (misaligned(stats, 16) || misaligned(y, 16)) return TR_ERR_ALIGN;
  if ((rc = check_ws(sh, ws, ws_bytes)) != TR_OK) return rc;
  SelectArgs a = select_args(in, sh, stats, d_k, d_k1, d_cu_k, idx, nullptr, h2, s, ws, d_status);
  cudaError_t err = launch_select_gather(a, y, static_cast<cudaStream_t>(stream), true);
  return err == cudaSuccess ? TR_OK : TR_ERR_CUDA;
}

tr_status tr_reduce(const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1, const int32_t *d_cu_k,
                    int32_t total_k, void *y, int32_t *idx, float *h2, float *s, void *ws, size_t ws_bytes,
                    int32_t *d_status, void *stream) {
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (total_k < 0 || total_k > sh.total) return TR_ERR_BUDGET;
  if (in->batch > 0 && (!d_k || !d_k1 || !d_cu_k || !idx || (total_k > 0 && !y))) return TR_ERR_ARG;
  if (misaligned(y, 16)) return TR_ERR_ALIGN;
  if ((rc = check_ws(sh, ws, ws_bytes)) != TR_OK) return rc;
  float *stats = reinterpret_cast<float *>(static_cast<char *>(ws) + ws_layout(sh.total).stats);
  rc = tr_score(in, stats, h2, s, stream);
  if (rc != TR_OK) return rc;
  if (in->cu_seqlens) {
    // Ragged batches: replicas of equal number per image would leave the
    // large images' copies to few CTAs; the grid-wide gather spreads them.
    rc = tr_select(in, stats, d_k, d_k1, d_cu_k, idx, nullptr, h2, s, ws, ws_bytes, d_status, stream);
    if (rc != TR_OK) return rc;
    return tr_gather(in, d_cu_k, idx, total_k, y, stream);
  }
  return tr_select_gather(in, stats, d_k, d_k1, d_cu_k, total_k, y, idx, h2, s, ws, ws_bytes, d_status, stream);
}

tr_status tr_gather(const tr_tokens *in, const int32_t *d_cu_k, const int32_t *idx, int32_t total_k, void *y,
                    void *stream) {
  return gather_impl(in, d_cu_k, idx, total_k, y, stream, true);
}

// ---------------------------------------------------------------- pipeline
struct tr_pipeline {
  cudaStream_t score_stream[TR_PIPELINE_MAX_SLOTS] = {}, select_stream = nullptr;
  int slots = 0;
  void *ws[TR_PIPELINE_MAX_SLOTS] = {};
  size_t ws_bytes = 0;
  cudaEvent_t scored[TR_PIPELINE_MAX_SLOTS] = {};
  cudaEvent_t done[TR_PIPELINE_MAX_SLOTS] = {};
  cudaEvent_t head[TR_PIPELINE_MAX_SLOTS] = {};  // the slot's batch scored
  long long submitted = 0;
  long long kernels = 0;  // kernels launched by the submissions
};

tr_status tr_pipeline_create(void *const *score_streams, void *select_stream, int32_t slots, void *const *ws,
                             size_t ws_bytes, tr_pipeline **out) {
  if (!out) return TR_ERR_ARG;
  *out = nullptr;
  if (slots < 1 || slots > TR_PIPELINE_MAX_SLOTS || !ws || !score_streams) return TR_ERR_ARG;
  for (int i = 0; i < slots; ++i)
    if (!ws[i] || misaligned(ws[i], 256)) return TR_ERR_WORKSPACE;
  tr_pipeline *p = new (std::nothrow) tr_pipeline;
  if (!p) return TR_ERR_ARG;
  for (int i = 0; i < slots; ++i) p->score_stream[i] = static_cast<cudaStream_t>(score_streams[i]);
  p->select_stream = static_cast<cudaStream_t>(select_stream);
  p->slots = slots;
  p->ws_bytes = ws_bytes;
  for (int i = 0; i < slots; ++i) {
    p->ws[i] = ws[i];
    if (cudaEventCreateWithFlags(&p->scored[i], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&p->done[i], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&p->head[i], cudaEventDisableTiming) != cudaSuccess) {
      tr_pipeline_destroy(p);
      return TR_ERR_CUDA;
    }
  }
  *out = p;
  return TR_OK;
}

tr_status tr_pipeline_submit(tr_pipeline *p, const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1,
                             const int32_t *d_cu_k, int32_t total_k, void *y, int32_t *idx, float *h2, float *s,
                             int32_t *d_status, void *score_begin, void *score_end) {
  if (!p) return TR_ERR_ARG;
  Shape sh;
  tr_status rc = check_tokens(in, &sh);
  if (rc != TR_OK) return rc;
  if (total_k < 0 || total_k > sh.total) return TR_ERR_BUDGET;
  if (in->batch > 0 && (!d_k || !d_k1 || !d_cu_k || !idx || (total_k > 0 && !y))) return TR_ERR_ARG;
  if (misaligned(y, 16) || misaligned(h2, 4) || misaligned(s, 4)) return TR_ERR_ALIGN;
  const int slot = (int)(p->submitted % p->slots);
  void *ws = p->ws[slot];
  if ((rc = check_ws(sh, ws, p->ws_bytes)) != TR_OK) return rc;
  float *stats = reinterpret_cast<float *>(static_cast<char *>(ws) + ws_layout(sh.total).stats);
  cudaStream_t a = p->score_stream[slot], b = p->select_stream;
  // The slot's workspace is free once the submission that used it last has
  // been selected and gathered.
  if (p->submitted >= p->slots && cudaStreamWaitEvent(a, p->done[slot], 0) != cudaSuccess) return TR_ERR_CUDA;
  // Consecutive batches' scoring may overlap (each slot has its score
  // stream): the next score kernel then fills the SMs the previous one frees
  // while it drains its last wave.  That pays while the last wave is a good
  // part of the kernel; for a long kernel (a batch of more than 20 waves of
  // rows) two interleaved score kernels only delay each other's selection,
  // so it waits for the previous batch's scoring instead.  (Measured on
  // GB300: 2 slots, llava576 169 us per step overlapped against 178 us
  // serial; ragged_dynres, 276k rows, 1072 us overlapped against 1017 us.)
  const long long wave_rows = (long long)kScoreWarps * 16 * sm_count();
  const int prev = (int)((p->submitted + p->slots - 1) % p->slots);
  if (sh.total > 20 * wave_rows && p->submitted > 0 && cudaStreamWaitEvent(a, p->head[prev], 0) != cudaSuccess)
    return TR_ERR_CUDA;
  // The caller's timing events become event-record nodes when the stream is
  // being captured into a graph (cudaEventRecordExternal, which is valid only
  // during a capture), so that they time each replay.
  cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
  if ((score_begin || score_end) && cudaStreamIsCapturing(a, &capturing) != cudaSuccess) return TR_ERR_CUDA;
  const unsigned rec_flags =
      capturing == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
  if (score_begin && cudaEventRecordWithFlags(static_cast<cudaEvent_t>(score_begin), a, rec_flags) != cudaSuccess)
    return TR_ERR_CUDA;
  if ((rc = tr_score(in, stats, h2, s, a)) != TR_OK) return rc;
  if (cudaEventRecord(p->head[slot], a) != cudaSuccess) return TR_ERR_CUDA;
  if (score_end && cudaEventRecordWithFlags(static_cast<cudaEvent_t>(score_end), a, rec_flags) != cudaSuccess)
    return TR_ERR_CUDA;
  if (cudaEventRecord(p->scored[slot], a) != cudaSuccess || cudaStreamWaitEvent(b, p->scored[slot], 0) != cudaSuccess)
    return TR_ERR_CUDA;
  if (d_status && cudaMemsetAsync(d_status, 0, TR_STATUS_WORDS * sizeof(int32_t), b) != cudaSuccess)
    return TR_ERR_CUDA;
  // At most a quarter of the SMs select at once (each CTA takes several
  // images in turn when the batch is larger): the rest keep scoring the
  // next batch at full bandwidth.  (Measured on GB300 against no cap and
  // caps of 1/2 and 1/8: best or equal on every workload; 256 per-frame
  // video images 198 us per step against 205 us uncapped.)
  const int sms = sm_count();
  const int cap = (sms + 3) / 4;
  // A uniform batch of one or two small images (up to 1024 tokens) selects
  // and gathers in one launch (tr_select_gather's replicas: the copy is split
  // over them and one kernel boundary leaves the step's critical path) when
  // the replicas stay within the same quarter of the SMs.  (Measured on
  // GB300: one 576-token image 21.9 -> 20.0 us per step; one 6272-token clip
  // 66 -> 74 us, its 16 replicas slowing one another, hence the size limit.)
  const int replicas = in->batch > 0 ? std::max(1, std::min(16, sms / in->batch)) : 0;
  if (!in->cu_seqlens && in->batch > 0 && in->n <= 1024 && in->batch * replicas <= cap) {
    SelectArgs a = select_args(in, sh, stats, d_k, d_k1, d_cu_k, idx, nullptr, h2, s, ws, d_status);
    if (launch_select_gather(a, y, b, false) != cudaSuccess) return TR_ERR_CUDA;
    p->kernels += (sh.total > 0) + 1;
  } else {
    if ((rc = select_capped(in, stats, d_k, d_k1, d_cu_k, idx, nullptr, h2, s, ws, p->ws_bytes, d_status, b, cap,
                            false)) != TR_OK)
      return rc;
    if ((rc = gather_impl(in, d_cu_k, idx, total_k, y, b, false)) != TR_OK) return rc;
    p->kernels += (sh.total > 0) + (in->batch > 0) + (total_k > 0);
  }
  if (cudaEventRecord(p->done[slot], b) != cudaSuccess) return TR_ERR_CUDA;
  ++p->submitted;
  return TR_OK;
}

tr_status tr_pipeline_wait(tr_pipeline *p, void *stream) {
  if (!p) return TR_ERR_ARG;
  const long long used = p->submitted < p->slots ? p->submitted : p->slots;
  for (long long i = 0; i < used; ++i)
    if (cudaStreamWaitEvent(static_cast<cudaStream_t>(stream), p->done[i], 0) != cudaSuccess) return TR_ERR_CUDA;
  return TR_OK;
}

long long tr_pipeline_kernels(const tr_pipeline *p) { return p ? p->kernels : 0; }

tr_status tr_pipeline_destroy(tr_pipeline *p) {
  if (!p) return TR_OK;
  for (int i = 0; i < TR_PIPELINE_MAX_SLOTS; ++i) {
    if (p->scored[i]) cudaEventDestroy(p->scored[i]);
    if (p->done[i]) cudaEventDestroy(p->done[i]);
    if (p->head[i]) cudaEventDestroy(p->head[i]);
  }
  delete p;
  return TR_OK;
}

}  // extern "C"
