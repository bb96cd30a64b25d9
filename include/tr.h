/*
 * tr.h -- C ABI of the ALTR visual-token reducer for GB300 (sm_103a).
 *
 * ALTR (arxiv 2607.13500, Section IV) keeps K of the N visual tokens of an
 * image: the K1 = floor(lambda K) tokens with the highest second-order Renyi
 * entropy of their channel-magnitude distribution (Stage I, Eq. 3-4), plus
 * K2 = K - K1 tokens taken at a fixed stride along the remaining tokens sorted
 * by the cosine between the final-layer MLP input x' and output x'' (Stage II,
 * Eq. 5-6), returned as X* = X_imp union X_div (Eq. 7, Algorithm 1).
 *
 * Conventions shared by every entry point:
 *  - Device pointers are owned by the caller; the library never allocates
 *    device memory, frees it or synchronises.  Every call enqueues work on
 *    `stream` (a cudaStream_t; NULL is the legacy default stream) and returns
 *    at once.  (A tr_pipeline owns host-side CUDA events, see below.)
 *  - Host-detectable errors (null or misaligned pointers, bad sizes, too small
 *    a workspace) are returned before anything is launched; outputs are left
 *    untouched.  A launch failure returns TR_ERR_CUDA.
 *  - Data-dependent conditions are counted in the optional device status
 *    words (int32[TR_STATUS_WORDS], accumulated with atomics; zero them before
 *    the call): [0] rows found to hold a non-finite value in an input the
 *    selection (or a requested H2 / s output) needed, [1] rows whose
 *    exact sums did not fit the exact representation (ordering of such a row
 *    falls back to its float key), [2] rows recomputed exactly to settle a
 *    near-tie, [3] images skipped because their budget was invalid
 *    (K < 0, K > N, K1 < 0 or K1 > K).
 *  - Kept indices are local to their image, ascending, and image b's
 *    occupy positions [cu_k[b], cu_k[b+1]) of `idx` and of `y`.
 *  - Ties go to the lower token index, in the top-K1 and in the sort.
 *  - The library keeps no global state besides two per-device caches (the
 *    "shared memory limit already raised" flags and the SM count, both
 *    atomic); calls from several host threads or on different streams may
 *    run concurrently when they use different workspaces and outputs.
 *  - The single-call entry points only enqueue kernels (no allocation,
 *    synchronisation or copies), so they can be captured into a CUDA graph
 *    and replayed; make one call on the device outside the capture first
 *    (it raises the kernels' shared-memory limit once).
 *  - tr_select, tr_gather, tr_select_gather and tr_reduce launch their
 *    kernels with programmatic dependent launch: a kernel may be scheduled
 *    while the kernel before it on the stream finishes, and waits in
 *    hardware for that kernel's completion before it reads anything, so
 *    stream order is kept (tr_score's kernel lets such a successor in as
 *    soon as all its CTAs run).  The pipeline launches normally.
 */
#ifndef TR_H
#define TR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  TR_OK = 0,
  TR_ERR_ARG = 1,         /* null pointer, negative or inconsistent size       */
  TR_ERR_BUDGET = 2,      /* K > N, lambda or ratio outside [0, 1] (host)      */
  TR_ERR_DTYPE = 3,       /* dtype not one of tr_dtype                         */
  TR_ERR_ALIGN = 4,       /* d * sizeof(elem) % 16 != 0 or a base not 16-B aligned */
  TR_ERR_WORKSPACE = 5,   /* workspace NULL, too small or not 256-B aligned    */
  TR_ERR_CUDA = 6,        /* a kernel launch failed                            */
  TR_ERR_UNSUPPORTED = 7  /* N_b > TR_MAX_N or d > TR_MAX_D                    */
} tr_status;

typedef enum { TR_F32 = 0, TR_BF16 = 1, TR_F16 = 2 } tr_dtype;

#define TR_MAX_N 16384        /* tokens per image (keys of one image stay in shared memory) */
#define TR_MAX_D 16384        /* channels per token                                  */
#define TR_STATS_WORDS 8      /* fp32 words of the per-row statistics record         */
#define TR_STATUS_WORDS 4

/*
 * The token tensors of a batch of images, packed row-major as [total, d]:
 * image b owns rows [cu_seqlens[b], cu_seqlens[b+1]) (ragged), or
 * [b*n, (b+1)*n) when cu_seqlens is NULL (uniform).
 */
typedef struct {
  const void *x;              /* visual tokens X, the Stage-I input and gather source (Sec. III-A) */
  const void *x_pre;          /* final-layer MLP input x' (Eq. 5); NULL means x' = x               */
  const void *x_post;         /* final-layer MLP output x'' (Eq. 5); required                      */
  int32_t dtype;              /* tr_dtype of all three tensors                                     */
  int32_t d;                  /* channels D                                                         */
  int32_t batch;              /* images B                                                           */
  int32_t n;                  /* tokens per image N when cu_seqlens is NULL                         */
  const int32_t *cu_seqlens;  /* device int32[batch+1] row offsets, or NULL                         */
  int32_t total;              /* total rows T (ragged: must equal cu_seqlens[batch])                */
  int32_t max_n;              /* ragged: max_b N_b (host-known); ignored when uniform              */
  int32_t flags;              /* selection options, 0 or TR_STRIDE_INTERVAL                         */
} tr_tokens;

/*
 * Positions of the diversity picks along X_rem sorted by s (M = |X_rem|):
 *   flags = 0:                  Algorithm 1, the integer stride
 *                               t = max(1, floor(M / K2)): 0, t, ..., (K2-1) t;
 *   flags = TR_STRIDE_INTERVAL: the fixed interval (N - |X_imp|) / K2 = M / K2
 *                               of Section IV-B taken as a real number:
 *                               floor(j M / K2) for j < K2.
 * Both pick K2 distinct positions; they agree whenever K2 divides M.
 */
#define TR_STRIDE_INTERVAL 1

/* Name of a status code (static string). */
const char *tr_status_string(int32_t status);

/* Library version string. */
const char *tr_version(void);

/*
 * Budgets of Algorithm 1, first step, and Eq. 7 (host only, no device work).
 * Per image b with N_b = h_seqlens[b] tokens:
 *   K_b  = k                          when k > 0,
 *        = max(1, floor(N_b r_num / r_den)) (0 if N_b = 0) when k <= 0;
 *   K1_b = floor(K_b lam_num / lam_den), K2_b = K_b - K1_b;
 *   h_cu_k[0] = 0, h_cu_k[b+1] = h_cu_k[b] + K_b.
 * lambda = lam_num / lam_den must lie in [0, 1] (the paper's split of K = 192
 * into 64 + 128 tokens, Section V-C, is lambda = 1/3).  Returns TR_ERR_BUDGET
 * when K_b > N_b, a ratio lies outside (0, 1] or lambda outside [0, 1];
 * TR_ERR_ARG for null pointers or batch < 0.  h_k, h_k1: int32[batch];
 * h_cu_k: int32[batch+1].
 */
tr_status tr_budgets(int32_t batch, const int32_t *h_seqlens, int32_t k, int32_t r_num, int32_t r_den,
                     int32_t lam_num, int32_t lam_den, int32_t *h_k, int32_t *h_k1, int32_t *h_cu_k);

/* Device workspace bytes that tr_select and tr_reduce need for `in`
 * (0 on invalid input).  The workspace must be 256-byte aligned. */
size_t tr_workspace_bytes(const tr_tokens *in);

/*
 * Scoring pass (Eq. 3, 4 and 6 for every token): one read of x, x', x''.
 *   stats: device fp32[total, TR_STATS_WORDS] (16-byte aligned), per row
 *          [0] L1 = sum_j |x_j|, [1] S2 = sum_j x_j^2, [2] A = sum_j x'_j^2,
 *          [3] B = sum_j x''_j^2, [4] P_hi, [5] P_lo with P = sum_j x'_j x''_j
 *          = P_hi + P_lo (double-float), [6] the importance key L1^2 / S2
 *          and [7] the consistency key P / sqrt(A B), both rounded once to
 *          fp32 and NaN when the row's sums left the fp32 error model
 *          (non-finite, or S2, A or B outside [2^-100, 2^100]).  L1, S2, A, B
 *          are fp32 sums of bounded rounding depth; P is accumulated
 *          error-free up to a ~1e-10 relative residue.
 *   h2:    device fp32[total] or NULL: H2 = -log sum_j p_j^2 = log(L1^2 / S2)
 *          (Eq. 3-4); 0 for an all-zero row.
 *   s:     device fp32[total] or NULL: s = P / sqrt(A B) (Eq. 6); 0 when
 *          x' or x'' is all zero.
 * h2 and s come from the fp32 sums; rows whose sums overflow fp32 (inputs
 * above ~2^63 in magnitude) or hold non-finite inputs get non-finite values
 * here and are settled exactly by tr_select / tr_reduce.
 */
tr_status tr_score(const tr_tokens *in, float *stats, float *h2, float *s, void *stream);

/*
 * Selection (Stage I top-K1, Stage II sort and stride pick, Algorithm 1)
 * from the statistics of tr_score.  Decisions are exact: keys whose float
 * bounds overlap are recomputed from the inputs in exact integer arithmetic,
 * so the result is the selection defined by the real-valued H2 and s with
 * the lower-index tie-break.
 *   d_k, d_k1:  device int32[batch] budgets K_b, K1_b (see tr_budgets).
 *   d_cu_k:     device int32[batch+1] prefix sums of K_b.
 *   idx:        device int32[cu_k[batch]] kept local indices (ascending).
 *   role:       device uint8[total] or NULL: 0 dropped, 1 X_imp, 2 X_div.
 *   h2, s:      device fp32[total] or NULL: when given, rows whose fp32 sums
 *               were unreliable (non-finite, overflowed or underflowed) and
 *               rows recomputed for a near-tie get H2 / s rewritten from the
 *               exact sums (-inf H2 / +inf s for non-finite inputs).
 *   ws:         device workspace of tr_workspace_bytes(in) bytes.
 *   d_status:   device int32[TR_STATUS_WORDS] or NULL.
 */
tr_status tr_select(const tr_tokens *in, const float *stats, const int32_t *d_k, const int32_t *d_k1,
                    const int32_t *d_cu_k, int32_t *idx, uint8_t *role, float *h2, float *s, void *ws,
                    size_t ws_bytes, int32_t *d_status, void *stream);

/*
 * Gather of the kept tokens (Eq. 7: X* holds the original token vectors):
 * y[r] = x[first row of image b + idx[r]] for cu_k[b] <= r < cu_k[b+1], a
 * bit copy of d elements in the input dtype.
 *   d_cu_k:   device int32[batch+1] prefix sums of K_b (as for tr_select).
 *   idx:      device int32[total_k] local kept indices (tr_select's output).
 *   total_k:  host int, = cu_k[batch].
 *   y:        device [total_k, d] in the input dtype, 16-byte aligned.
 * A row whose index falls outside its image's tokens is written as zeros.
 */
tr_status tr_gather(const tr_tokens *in, const int32_t *d_cu_k, const int32_t *idx, int32_t total_k, void *y,
                    void *stream);

/*
 * Selection and gather in one launch, from the statistics of tr_score: the
 * result of tr_select (idx, optional H2 / s fix-ups, status) plus the kept
 * rows y as tr_gather would copy them.  When there are fewer images than
 * SMs, each image's selection is run by several CTAs at once and each copies
 * its share of the kept rows (the selection is deterministic, so all reach
 * the same indices; only one writes idx and the status words).
 *   total_k:  host int, = cu_k[batch]; y: device [total_k, d], 16-byte aligned.
 *   Other arguments as in tr_select (role is not produced).
 */
tr_status tr_select_gather(const tr_tokens *in, const float *stats, const int32_t *d_k, const int32_t *d_k1,
                           const int32_t *d_cu_k, int32_t total_k, void *y, int32_t *idx, float *h2, float *s,
                           void *ws, size_t ws_bytes, int32_t *d_status, void *stream);

/*
 * The whole path in one call on `stream`, with the statistics kept in the
 * workspace: tr_score then tr_select_gather for a uniform batch (two kernel
 * launches); tr_score, tr_select and tr_gather for a ragged one (three).
 *   total_k:  host int, = cu_k[batch] (the number of output rows).
 *   y:        device [total_k, d] in the input dtype, 16-byte aligned.
 *   idx, h2, s, d_status: as in tr_select (role is not produced); h2 and s
 *             may be NULL.
 */
tr_status tr_reduce(const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1, const int32_t *d_cu_k,
                    int32_t total_k, void *y, int32_t *idx, float *h2, float *s, void *ws, size_t ws_bytes,
                    int32_t *d_status, void *stream);

/*
 * tr_reduce without a caller-provided workspace, for callers that cannot
 * allocate device memory (code running inside a host framework whose
 * allocator it cannot reach, plugins or callbacks that must not call
 * cudaMalloc, loops that must not allocate once they run).  The paper has
 * no counterpart: this is a deployment convenience of this library.
 *
 * Same arguments and results as tr_reduce, minus ws / ws_bytes.  Its scratch
 * is a device array of TR_NOALLOC_SCRATCH_BYTES bytes inside libtr, present
 * on every GPU that loads the library until the process exits; batches of
 * more than TR_NOALLOC_MAX_ROWS token rows are rejected with
 * TR_ERR_UNSUPPORTED.  The call allocates nothing.  The first call on a
 * device looks up that array's device address (with the device current),
 * so make the first call on each device before any stream capture.  All
 * calls share the array: calls whose work may overlap on the GPU race and
 * must be serialised by the caller.
 */
#define TR_NOALLOC_MAX_ROWS 32768
#define TR_NOALLOC_SCRATCH_BYTES (8u << 20)
tr_status tr_reduce_noalloc(const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1, const int32_t *d_cu_k,
                            int32_t total_k, void *y, int32_t *idx, float *h2, float *s, int32_t *d_status,
                            void *stream);

/*
 * Overlapped reduction of successive batches, a stream pipeline over `slots`
 * slots.  Submission i uses slot i mod slots: it scores its batch on
 * score_streams[slot] (tr_score), then selects (tr_select) and gathers
 * (tr_gather) it on `select_stream`, which waits for that scoring only (a
 * uniform batch of one or two images of at most 1024 tokens is selected and
 * gathered by one tr_select_gather launch instead).  So
 * the selection and gather of one batch run while the next batch is scored,
 * and with a score stream per slot one batch's scoring starts while the
 * previous score kernel drains.  Give `select_stream` the higher priority:
 * the score kernel's CTAs retire one by one, and a higher-priority kernel
 * takes the SMs they free.  The slot's workspace ws[slot] (ws_bytes >=
 * tr_workspace_bytes bytes, 256-byte aligned, owned by the caller) is reused
 * only after the submission that used it last has been gathered (the score
 * stream waits for it).
 *
 * Ordering the caller keeps: the inputs of a submission (x, x', x'') stay
 * unchanged, and its outputs (y, idx, h2, s, d_status) untouched by other
 * work, until select_stream has passed the submission -- give each
 * submission still in flight its own output buffers (one set per slot).
 * Work that consumes a submission's outputs orders itself after it on
 * select_stream (or tr_pipeline_wait).
 *
 * The pipeline owns 3 x slots CUDA events, created on the current device by
 * tr_pipeline_create (make it the device of every stream) and destroyed by
 * tr_pipeline_destroy; it allocates no device memory and never synchronises.
 * One host thread at a time may submit to a pipeline (it keeps a count).
 *   tr_pipeline_create: score_streams holds `slots` cudaStream_t (they may
 *     repeat one stream); ws holds `slots` workspaces.
 *   tr_pipeline_submit: arguments as in tr_reduce, except that d_status is
 *     zeroed by the call itself (on select_stream, before the selection);
 *     score_begin / score_end are optional cudaEvent_t (or NULL) recorded on
 *     the slot's score stream right before and after the score kernel, to
 *     time it (as event-record nodes when the stream is being captured).
 *     Host-detectable errors are returned before anything is enqueued.
 *   tr_pipeline_wait: makes `stream` wait for every submission so far.
 *   tr_pipeline_kernels: kernels launched by the submissions so far (three
 *     per submission -- score, select, gather -- or two when a tiny uniform
 *     batch is selected and gathered in one launch); 0 for NULL.
 *
 * Graph capture: submissions made while the streams are captured into a
 * CUDA graph (forked from the capturing stream, joined back with
 * tr_pipeline_wait and a wait on each score stream) become one graph whose
 * replay runs those steps, overlapped as above, with a single launch.  Use a
 * pipeline created for the capture (no submission before it: the first
 * `slots` submissions of a pipeline wait on no earlier event) and only
 * replay it afterwards.
 */
#define TR_PIPELINE_MAX_SLOTS 8
typedef struct tr_pipeline tr_pipeline;
tr_status tr_pipeline_create(void *const *score_streams, void *select_stream, int32_t slots, void *const *ws,
                             size_t ws_bytes, tr_pipeline **out);
tr_status tr_pipeline_submit(tr_pipeline *p, const tr_tokens *in, const int32_t *d_k, const int32_t *d_k1,
                             const int32_t *d_cu_k, int32_t total_k, void *y, int32_t *idx, float *h2, float *s,
                             int32_t *d_status, void *score_begin, void *score_end);
tr_status tr_pipeline_wait(tr_pipeline *p, void *stream);
long long tr_pipeline_kernels(const tr_pipeline *p);
tr_status tr_pipeline_destroy(tr_pipeline *p);

/*
 * ---- The encoder's final-layer MLP with the scoring fused in (Eq. 5) ----
 *
 * Section IV-B takes x' (the input of the vision encoder's last MLP) and
 * x'' = f(x') = W2 sigma(W1 x') (its output, Eq. 5) from the encoder's
 * forward pass.  These two calls run that MLP on the tensor cores, and the
 * second one scores every token in its epilogue, so the selection needs no
 * separate pass over x, x', x'':
 *
 *   tr_mlp_hidden:  H = sigma(x' W1^T + b1)                       [t, d_hidden]
 *   tr_mlp_score:   x'' = H W2^T + b2, rounded to bf16 and stored  [t, d]
 *                   x   = resid + x'' (the block's output tokens X, the
 *                         Stage-I input and gather source), rounded to bf16
 *                         and stored; x = x'' when resid is NULL
 *                   stats: the per-row record of tr_score, with its sums
 *                         taken over the stored x, x' and x''.
 *
 * tr_select (or tr_select_gather) then takes tokens {x, x', x''} and these
 * stats exactly as it takes tr_score's; the result is the selection defined
 * by the stored tensors.  The sums of each record carry less rounding than
 * tr_score's (every term enters through TwoSum), within the same
 * certification bounds.
 *
 * Operands and outputs are bf16, row-major, 16-byte aligned; d and d_hidden
 * are multiples of 16.  Accumulation is fp32 in tensor memory; sigma is
 * evaluated in fp32 on the accumulator plus b1 and rounded once to bf16.
 * d_error (optional device int32, zero it first) gets a non-zero bit when a
 * pipeline wait inside the kernel timed out (not expected in a correct run;
 * the kernel then stops early and its outputs are incomplete).
 */
#define TR_ACT_GELU 0        /* x Phi(x), the erf form                        */
#define TR_ACT_QUICK_GELU 1  /* x / (1 + exp(-1.702 x)), CLIP's variant        */
#define TR_ACT_NONE 2
#define TR_MLP_MAX_HIDDEN 65536
typedef struct {
  const void *x_pre;   /* [t, d] bf16: the MLP input x' (Eq. 5)                        */
  const void *resid;   /* [t, d] bf16 added to x'' to form x, or NULL (x = x'')        */
  const void *w1;      /* [d_hidden, d] bf16 (nn.Linear layout)                        */
  const void *w2;      /* [d, d_hidden] bf16                                           */
  const float *b1;     /* [d_hidden] fp32 or NULL                                      */
  const float *b2;     /* [d] fp32 or NULL                                             */
  int32_t t;           /* rows (tokens of the whole batch)                              */
  int32_t d;           /* channels D                                                    */
  int32_t d_hidden;    /* hidden width of the MLP                                       */
  int32_t act;         /* sigma: TR_ACT_GELU, TR_ACT_QUICK_GELU or TR_ACT_NONE          */
} tr_mlp;

/* H = sigma(x' W1^T + b1): h is device bf16 [t, d_hidden]. */
tr_status tr_mlp_hidden(const tr_mlp *m, void *h, int32_t *d_error, void *stream);

/* Scratch bytes of tr_mlp_score (256-byte aligned device memory); 0 on invalid input. */
size_t tr_mlp_workspace_bytes(const tr_mlp *m);

/*
 * x'' = H W2^T + b2 and x = resid + x'' (both stored, bf16 [t, d]) with the
 * scoring of every row in the same pass: stats is device fp32
 * [t, TR_STATS_WORDS] laid out as in tr_score, h2 / s optional fp32 [t].
 * x_post and x must not overlap the inputs.
 */
tr_status tr_mlp_score(const tr_mlp *m, const void *h, void *x_post, void *x, float *stats, float *h2, float *s,
                       void *ws, size_t ws_bytes, int32_t *d_error, void *stream);

/*
 * ---- The first projector layer on the kept tokens, gathered on the fly ----
 *
 * The projector P maps the kept tokens X* = X_imp union X_div (Eq. 7) into
 * the LLM's embedding space (Z* = P(X*), Section III-A).  This call runs its
 * first layer, z = sigma(X* W^T + bias), on the tensor cores with the rows of
 * X* read straight from x by the selection's kept indices, so the gathered
 * copy y (tr_gather) is not needed for it:
 *   in:       the tokens x (bf16, as given to tr_select; x_pre / x_post unused)
 *   d_cu_k:   device int32[batch+1] prefix sums of K_b; idx: device int32
 *             [total_k] kept local indices (tr_select's output)
 *   w:        device bf16 [d_out, d] (nn.Linear layout); bias fp32 [d_out] or NULL
 *   act:      TR_ACT_GELU (LLaVA-1.5's projector), TR_ACT_QUICK_GELU, TR_ACT_NONE
 *   z:        device bf16 [total_k, d_out], row r for kept slot r
 * An index outside its image's tokens gives a row of zeros as input.  d and
 * d_out are multiples of 16; pointers 16-byte aligned.  d_error as for
 * tr_mlp_hidden.  Further projector layers are plain GEMMs on z.
 */
tr_status tr_project_kept(const tr_tokens *in, const int32_t *d_cu_k, const int32_t *idx, int32_t total_k,
                          const void *w, const float *bias, int32_t d_out, int32_t act, void *z, int32_t *d_error,
                          void *stream);

/*
 * The same first projector layer (Section III-A) on rows already gathered --
 * tr_gather's y, or any dense rows:
 *   y:        device bf16 [rows, d]
 *   w, bias, d_out, act: as for tr_project_kept
 *   z:        device bf16 [rows, d_out], row r from y's row r
 * z = sigma(y W^T + bias) by the kernel of tr_mlp_hidden; for y = the rows
 * that tr_project_kept reads, the two give the same z bit for bit (the same
 * MMA order and epilogue arithmetic).  Gathering first and projecting the
 * dense rows is the faster route on GB300: tr_project_kept's row loads are
 * TMA gathers whose issue rate sets its pace, while the copy costs one write
 * and one read of rows * d * 2 bytes.  d and d_out multiples of 16, pointers
 * 16-byte aligned; rows = 0 does nothing.  d_error as for tr_mlp_hidden.
 */
tr_status tr_project(const void *y, int32_t rows, int32_t d, const void *w, const float *bias, int32_t d_out,
                     int32_t act, void *z, int32_t *d_error, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* TR_H */
