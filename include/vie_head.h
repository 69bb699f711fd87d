/*
 * vie_head.h - C ABI of the exact LLM output head for GB300 (sm_103a).
 *
 * The head computes, for each decode query h (paper, Section 3):
 *     z = W_out h,            z_i = <w_i, h>        (W_out: V rows of width d)
 * selects the k rows with the largest z_i (exhaustive maximum inner product
 * search, Sections 2-3) and can write those k logits into a full-vocabulary
 * tensor that is -infinity everywhere else (Section 3, the sparse logit
 * tensor handed to standard logit processors).
 *
 * Conventions shared by every call:
 *   - Pointers marked "device" are CUDA device pointers of the device that is
 *     current on the calling thread; "host" pointers are ordinary memory.
 *   - A vie_stream is a cudaStream_t (NULL = the legacy default stream).  Calls
 *     that take a stream are asynchronous on it: they validate on the host,
 *     enqueue kernels and return without synchronising.
 *   - Every call returns a vie_status.  On anything but VIE_OK,
 *     vie_last_error() returns a message for the calling thread.  Argument
 *     errors are detected on the host before anything is enqueued; they leave
 *     no CUDA error behind.
 *   - Device-side problems (an out-of-range scatter index, a pipeline wait
 *     that ran past its time limit) never trap: the kernel records a flag and
 *     returns, and the next vie_device_status / vie_head_device_status call
 *     reports VIE_ERR_DEVICE.  The outputs of the call that recorded a wait
 *     time-out are unspecified (every write still stays inside them).
 *   - Logits are fp32.  Ranking is by logit descending; equal logits are
 *     ranked by ascending vocabulary index, and -0.0 ranks as +0.0 (and is
 *     returned as +0.0).  Inputs must be finite; results for NaN or infinite
 *     inputs are unspecified.
 */
#ifndef VIE_HEAD_H
#define VIE_HEAD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct vie_head vie_head; /* opaque handle */
typedef void *vie_stream;         /* a cudaStream_t */

typedef enum {
    VIE_OK = 0,
    VIE_ERR_INVALID_ARG = 1, /* a pointer, size or enum value is out of range */
    VIE_ERR_UNSUPPORTED = 2, /* valid request beyond what this library serves */
    VIE_ERR_CUDA = 3,        /* a CUDA runtime call or a launch failed        */
    VIE_ERR_OOM = 4,         /* device memory could not be allocated          */
    VIE_ERR_DEVICE = 5       /* a kernel recorded a device-side problem       */
} vie_status;

typedef enum { VIE_DTYPE_BF16 = 0 } vie_dtype;

/* Limits of this library. */
#define VIE_K_MAX 1024     /* largest k of vie_head_topk                    */
#define VIE_BATCH_MAX 1024 /* largest batch of vie_head_topk                */
#define VIE_D_MAX 16384    /* largest hidden size d                         */
#define VIE_MANY_MAX (1 << 24)     /* largest n of vie_head_topk_many       */
#define VIE_RECALL_N_MAX (1 << 28) /* largest n of vie_recall_hits          */
#define VIE_RECALL_M_MAX (1 << 20) /* largest candidate count m             */

/* Read-only facts about a handle (for callers that size buffers or report). */
typedef struct {
    int64_t V;            /* vocabulary rows                                 */
    int32_t d;            /* hidden size                                     */
    int32_t d_pad;        /* row pitch in elements: d rounded up to 8        */
    int32_t ctas;         /* CTAs of one projection launch (one per SM max)  */
    int32_t device;       /* CUDA device ordinal the handle lives on         */
    int64_t weight_bytes; /* bytes of the owned padded copy of W_out         */
    int64_t scratch_bytes;/* bytes of per-handle scratch                      */
} vie_head_props;

/*
 * vie_head_create - take a copy of W_out in the layout the kernels stream.
 * Section 3 treats the rows of W_out as a static database that is prepared
 * once and reused for every query; this is that preparation step.
 *
 *   W_out  device, bf16 (raw bit patterns), row-major [V, d], any alignment
 *          of 2 bytes.  Only read during the call; the caller may free it
 *          afterwards.
 *   V      1 <= V <= 2^31 - 2;   d   1 <= d <= VIE_D_MAX;
 *   dtype  VIE_DTYPE_BF16 (the only dtype of this library).
 *   out    host; receives the new handle.
 *
 * The handle owns a padded copy [V, d_pad] (d_pad = d rounded up to a
 * multiple of 8, pad = +0) plus its scratch.  The copy runs on the legacy
 * default stream of the current device and the call returns after the device
 * has finished it.  Errors: VIE_ERR_INVALID_ARG (null pointer, bad size,
 * W_out not device memory of the current device), VIE_ERR_UNSUPPORTED
 * (dtype), VIE_ERR_OOM, VIE_ERR_CUDA.
 */
vie_status vie_head_create(const void *W_out, int64_t V, int32_t d, vie_dtype dtype,
                           vie_head **out);

/*
 * vie_head_create_e4m3 - a head whose rows are stored as 8-bit floats: the
 * paper names weight quantisation as a bandwidth saving orthogonal to its
 * method (Section 4); this is that variant of the exact head, streaming half
 * the bytes of the bf16 head per decode step.
 *
 *   W_out   device, bf16, row-major [V, d], 2-byte aligned (as for
 *           vie_head_create); quantised on the device before the call returns.
 *   V, d    as for vie_head_create.
 *
 * Row i is stored as e4m3 codes (1 sign, 4 exponent bits with bias 7, 3
 * mantissa bits, largest finite value 448) and one fp32 scale:
 *   scale_i = max_j |w_ij| / 448 in fp32 (1 for an all-zero row);
 *   q_ij = w_ij / scale_i in fp32, rounded to the nearest e4m3 value (ties
 *          to even, saturated at +-448);
 * and every top-k call on the handle (vie_head_topk, _sparse, _host,
 * _sample) computes z_i = scale_i * sum_j e4m3(q_ij) * h_j with fp32
 * accumulation, then the same exact top-k.  Calls with k <= 128 on rows of
 * at least 128 codes run on the tensor cores (tcgen05 kind::f8f6f4; each
 * query enters as four e4m3 pieces with power-of-two scales, which keep it to
 * within 2^-16 |h_j| per entry), from batch 1 (vie_head_plan reports path
 * 1); other calls use the streaming CUDA-core kernel.  Same errors as
 * vie_head_create.
 */
vie_status vie_head_create_e4m3(const void *W_out, int64_t V, int32_t d, vie_head **out);

/* Copies an e4m3 handle's codes (device uint8 [V, d], row-major) and scales
 * (device fp32 [V]) to caller buffers, asynchronously on `stream`.
 * VIE_ERR_INVALID_ARG for a bf16 handle or NULL arguments. */
vie_status vie_head_export_e4m3(const vie_head *head, uint8_t *codes, float *scales,
                                vie_stream stream);

/* Frees the padded copy and the scratch.  NULL is accepted.  The caller must
 * make sure no work using the handle is still running (synchronise first). */
vie_status vie_head_destroy(vie_head *head);

/* Fills *props (host) with the handle's facts. */
vie_status vie_head_get_props(const vie_head *head, vie_head_props *props);

/* How a vie_head_topk / vie_head_topk_sparse call of this size runs. */
typedef struct {
    int32_t path;     /* 0: streaming CUDA-core kernel, 1: tensor-core kernel  */
    int32_t groups;   /* query groups, one pass over W_out each               */
    int32_t launches; /* kernel launches the call enqueues                    */
} vie_topk_plan;

/* Fills *plan (host) for a call with this batch and k; the same argument
 * checks as vie_head_topk.  Nothing is enqueued. */
vie_status vie_head_plan(const vie_head *head, int32_t batch, int32_t k, vie_topk_plan *plan);

/*
 * Launch options - a hook for tests and tuning; the paper has no counterpart.
 *
 * By default the path and launch shape of a call depend only on the call
 * (batch, k), the handle (V, d, bf16 or e4m3 rows) and the device: the
 * defaults below are the shapes that measured fastest on GB300 and that the
 * test suite covers.  An option changes how the work is laid out (which
 * kernel, stage sizes, work split), never the results: every setting gives
 * the same top-k under the same ranking rule.  Options are process-wide
 * (all handles, all threads) and are read when a call plans its launches, so
 * a change takes effect from the next call on; change them only while no
 * other thread is inside a call of this library.  Nothing is read from the
 * environment.
 */
typedef enum {
    VIE_OPT_STAGE_MIN_KB = 0,      /* smallest streaming weight stage, KB       (48)  */
    VIE_OPT_STATIC_PCT = 1,        /* % of W's pieces dealt round robin, rest
                                      drawn from a shared pool                   (85)  */
    VIE_OPT_POOL_DIV = 2,          /* pool pieces = one stage / this, 1..64      (1)   */
    VIE_OPT_TC_MIN_BATCH = 3,      /* smallest batch of a bf16 head sent to the
                                      tensor cores (k <= 128)                   (2)   */
    VIE_OPT_TC_KPS = 4,            /* most K-blocks per tensor-core stage, 1..4  (4)   */
    VIE_OPT_TC_MIN_BATCH_E4M3 = 5, /* the same threshold for e4m3 heads          (1)   */
    VIE_OPT_HALF_ROWS = 6,         /* streaming projection, one row per
                                      half-warp: 1 on, 0 off, -1 automatic       (-1)  */
    VIE_OPT_HOST_H_DIRECT = 7,     /* vie_head_topk_host reads page-locked
                                      queries in place: 1, or copies them: 0     (1)   */
    VIE_OPT_EARLY_MERGE = 8,       /* single-query streaming launches with
                                      k <= 64: one CTA merges the per-CTA lists
                                      while the others still stream: 1, or the
                                      last CTA to finish merges them all: 0      (1)   */
    VIE_OPT_COUNT = 9
} vie_launch_option;

#define VIE_OPT_DEFAULT INT32_MIN /* value that restores an option's default */

/* Sets one option (VIE_OPT_DEFAULT restores its default).  Errors:
 * VIE_ERR_INVALID_ARG for an unknown option or a value outside the range
 * given above (the option keeps its value). */
vie_status vie_set_launch_option(vie_launch_option option, int32_t value);

/* Reads one option's current value into *value (host). */
vie_status vie_get_launch_option(vie_launch_option option, int32_t *value);

/*
 * vie_head_topk - exact top-k of z = W_out h for a batch of queries
 * (Section 3: output projection followed by top-k selection, computed by
 * exhaustive MIPS over every row, Section 2).
 *
 *   h           device, fp32, row-major [batch, d] (4-byte aligned).
 *   batch       1 <= batch <= VIE_BATCH_MAX.
 *   k           1 <= k <= min(V, VIE_K_MAX).
 *   out_idx     device, int32 [batch, k]: vocabulary indices, best first.
 *   out_logits  device, fp32  [batch, k]: their logits (fp32 accumulation of
 *               the bf16 x fp32 products).
 *   stream      the stream the work is enqueued on.
 *
 * The full logit vector is never written to memory.  Calls using the same
 * handle share its scratch, so at most one vie_head_topk per handle may be
 * in flight at a time (calls on one stream are naturally serialised).
 * No allocation and no host synchronisation happen inside the call.
 * Errors: VIE_ERR_INVALID_ARG, VIE_ERR_CUDA (launch failure).
 */
vie_status vie_head_topk(vie_head *head, const float *h, int32_t batch, int32_t k,
                         int32_t *out_idx, float *out_logits, vie_stream stream);

/*
 * vie_head_topk_sparse - vie_head_topk and the sparse full-vocabulary logit
 * tensor of Section 3 in one launch: besides out_idx / out_logits it writes
 *   out_sparse  device, fp32 [batch, V] (4-byte aligned): -inf (0xFF800000)
 *               everywhere except out_sparse[b, out_idx[b, j]] =
 *               out_logits[b, j] (the same bits).
 * The result equals vie_head_topk followed by vie_scatter_sparse_logits on
 * its outputs.  Same limits, sharing rule and errors as vie_head_topk.
 */
vie_status vie_head_topk_sparse(vie_head *head, const float *h, int32_t batch, int32_t k,
                                int32_t *out_idx, float *out_logits, float *out_sparse,
                                vie_stream stream);

/*
 * vie_head_topk_host - one whole decode step for a caller whose queries and
 * results live in host memory: copies h in, runs vie_head_topk_sparse (or
 * vie_head_topk when out_sparse is NULL), copies the top-k out and waits for
 * it.  The paper has no counterpart: it is the end-to-end form of the call.
 *
 *   h_host       host, fp32, row-major [batch, d].  Page-locked memory
 *                (cudaMallocHost / cudaHostRegister) keeps the copies
 *                asynchronous; pageable memory works, staged by the driver.
 *   idx_host     host, int32 [batch, k];  logits_host  host, fp32 [batch, k].
 *   out_sparse   device, fp32 [batch, V] (4-byte aligned), or NULL.
 *   batch, k, stream: as for vie_head_topk.
 *
 * Page-locked buffers (mapped into the device's address space) are used in
 * place: the kernels read page-locked queries straight from host memory, and
 * when idx_host and logits_host are both page-locked the kernel that merges
 * the top-k writes it there, with no copies.  Other buffers pass through
 * device buffers owned by the handle:
 * allocated by the first call that needs them (larger ones by a later call
 * that needs more, VIE_ERR_OOM if that fails), freed by vie_head_destroy.  The
 * call synchronises `stream` before it returns, so the host outputs are
 * ready; a device-side problem is reported by the next
 * vie_head_device_status, as for vie_head_topk.  At most one call per handle
 * at a time, as for vie_head_topk.
 */
vie_status vie_head_topk_host(vie_head *head, const float *h_host, int32_t batch, int32_t k,
                              int32_t *idx_host, float *logits_host, float *out_sparse,
                              vie_stream stream);

/*
 * vie_sample_topk - top-k sampling on the k candidates of each query
 * (Section 2: top-k sampling draws the next token from the k most probable
 * tokens; Section 3: top-p and min-p act as a second stage on the retrieved
 * logits; Section 4 samples with k = 50).  Per query, in fp32:
 *   p_j = softmax of logits[j] / temperature over the k candidates;
 *   top-p keeps the shortest prefix whose probability reaches top_p (at
 *   least one candidate); min-p keeps the candidates with p_j >= min_p * p_0;
 *   the kept set is the shorter prefix of the two;
 *   the token is the first kept candidate j whose cumulative probability
 *   exceeds u * (kept mass), where u in [0, 1) is the top 24 bits of the first
 *   output word of Philox4x32-10 (Salmon et al., SC 2011) at counter
 *   (step low, step high, query, 0) with key (seed low, seed high), times
 *   2^-24: the same (seed, step) gives the same draws, a new step new ones.
 *
 *   idx, logits  device, int32 / fp32 [batch, k]: candidates sorted by logit,
 *                best first, as vie_head_topk returns them (4-byte aligned).
 *   batch >= 1;  1 <= k <= VIE_K_MAX.
 *   temperature  > 0 and finite;  0 < top_p <= 1;  0 <= min_p <= 1.
 *   out_token    device, int32 [batch]: the drawn vocabulary index.
 *   out_prob     device, fp32 [batch]: its probability among the kept
 *                candidates.
 *   stream       the stream the work is enqueued on.
 *
 * The launch may start while the previous kernel on the stream finishes
 * (programmatic dependent launch); it reads idx and logits only after that
 * kernel has completed.  No allocation, no sync.
 */
vie_status vie_sample_topk(const int32_t *idx, const float *logits, int32_t batch, int32_t k,
                           float temperature, float top_p, float min_p, uint64_t seed,
                           uint64_t step, int32_t *out_token, float *out_prob, vie_stream stream);

/*
 * vie_head_topk_sample - vie_head_topk_sparse (or vie_head_topk when
 * out_sparse is NULL) followed by vie_sample_topk on its output: the whole
 * decode-step head with the next token drawn on the device.  Arguments as for
 * those two calls; k <= VIE_K_MAX.
 */
vie_status vie_head_topk_sample(vie_head *head, const float *h, int32_t batch, int32_t k,
                                float temperature, float top_p, float min_p, uint64_t seed,
                                uint64_t step, int32_t *out_idx, float *out_logits,
                                float *out_sparse, int32_t *out_token, float *out_prob,
                                vie_stream stream);

/*
 * vie_head_topk_many - the exact top-k of many hidden states, e.g. as the
 * ground truth against which an approximate head's Recall@k is measured
 * (Section 4.3 measures it over 20k hidden states).  The same results as
 * vie_head_topk on each block of up to VIE_BATCH_MAX consecutive states,
 * enqueued one block after the other on `stream`.
 *
 *   h          device, fp32 [n, d], row-major (4-byte aligned).
 *   n          1 <= n <= VIE_MANY_MAX;   k as for vie_head_topk.
 *   out_idx, out_logits  device, int32 / fp32 [n, k].
 *
 * Errors as for vie_head_topk; a block that fails to launch stops the call
 * (earlier blocks stay enqueued).
 */
vie_status vie_head_topk_many(vie_head *head, const float *h, int64_t n, int32_t k,
                              int32_t *out_idx, float *out_logits, vie_stream stream);

/*
 * vie_recall_hits - Recall@k bookkeeping (Section 4.3: recall is the share
 * of the exact head's top-k tokens that an approximate search also
 * retrieves).  For each query q:
 *   out_hits[q] = #{ j < k : exact[q, j] >= 0 and exact[q, j] is among
 *                            approx[q, 0], ..., approx[q, m - 1] },
 * the candidates taken as a set (a repeated candidate counts once) and
 * negative candidates as empty slots.  Recall@k over the n queries is
 * sum(out_hits) / (n k).  Integer work: the counts are exact.
 *
 *   exact     device, int32 [n, k]: the exact top-k indices (vie_head_topk,
 *             vie_head_topk_many).
 *   approx    device, int32 [n, m]: the approximate method's candidates.
 *   1 <= n <= VIE_RECALL_N_MAX;  1 <= k <= VIE_K_MAX;  1 <= m <= VIE_RECALL_M_MAX.
 *   out_hits  device, int32 [n].  All buffers 4-byte aligned.
 *
 * Asynchronous on `stream`, launched as a programmatic dependent of the
 * kernel before it (it reads its inputs only after that kernel completed).
 * Errors: VIE_ERR_INVALID_ARG (NULL, sizes, alignment), VIE_ERR_CUDA.
 */
vie_status vie_recall_hits(const int32_t *exact, int32_t k, const int32_t *approx, int32_t m,
                           int64_t n, int32_t *out_hits, vie_stream stream);

/*
 * vie_scatter_sparse_logits - the sparse full-vocabulary logit tensor of
 * Section 3: out[b, v] = -inf (bit pattern 0xFF800000) for every v, then
 * out[b, idx[b, j]] = logits[b, j] for j < k (values copied bit for bit).
 *
 *   idx     device, int32 [batch, k];   logits  device, fp32 [batch, k].
 *   batch   >= 1;  k >= 1;  V >= 1.
 *   out     device, fp32 [batch, V] (4-byte aligned).
 *
 * Indices within a row are expected to be distinct; if they repeat, which
 * value lands is unspecified.  An index outside [0, V) is skipped and sets
 * the device flag reported by vie_device_status.  No allocation, no sync.
 */
vie_status vie_scatter_sparse_logits(const int32_t *idx, const float *logits, int32_t batch,
                                     int32_t k, int64_t V, float *out, vie_stream stream);

/*
 * vie_head_topk_noalloc - vie_head_topk for callers that cannot allocate
 * device memory.  The paper has no counterpart: this is a deployment variant.
 *
 * Some callers are not allowed to call cudaMalloc at all: serving engines
 * whose device memory is carved out of one budget up front (a further
 * allocation could fail mid-request or take memory another model was
 * promised), and latency-critical decode loops that cannot afford the
 * implicit device synchronisation an allocation may bring.  A vie_head
 * allocates its padded weight copy and scratch in vie_head_create, so those
 * callers cannot make one.  This entry point takes the weights as they are
 * and keeps its scratch in a fixed array compiled into the library instead.
 *
 *   W_out       device memory of the current device (or managed memory),
 *               bf16 bit patterns, row-major [V, d], 16-byte aligned, d a
 *               multiple of 8 (rows must already be 16-byte vectors).
 *   V, d        1 <= V <= 2^31 - 2;  8 <= d <= VIE_D_MAX.
 *   h, batch, k, out_idx, out_logits, stream: as for vie_head_topk.
 *
 * Every batch runs on the streaming CUDA-core kernel, in query groups of up
 * to `cap` queries, one launch per group:
 *   cap = 8, halved (not below 1) while cap * d * 4 > 65536 or, for k > 64,
 *         while cap * c * 8 > 32768, where c = max(256, 2k rounded up to a
 *         multiple of 64) is the candidate buffer of one query.
 * Scratch: one 1 MiB array per device (every GPU that loads the library keeps
 * it until the process exits), of which the first 256 bytes hold counters.
 * A call needs
 *   8 * (round_up_even(slots * ctas * k) + slots * ctas * 8)
 * bytes of the rest, where ctas = min(SM count, ceil(V / 64), 1024) and
 * slots = the batch rounded up to a power of two, at most cap; larger
 * requests return VIE_ERR_UNSUPPORTED with the sizes in the message.  Groups
 * of one call run one after the other on `stream` and reuse the same lists
 * (the kernel re-arms its counters at the end of each launch).  The call clears
 * the counters at the start of the array with cudaMemsetAsync on `stream`
 * and allocates nothing (no cudaMalloc, no cudaFree, no allocating library
 * routine).
 * The first call on a device looks up the array's device address with
 * cudaGetSymbolAddress (once per device); make that first call before any
 * stream capture.  Every call shares the one array, so calls whose work
 * overlaps on the GPU (other streams, other threads) race and corrupt each
 * other's results: serialise them.  Device-side problems set the flag read by
 * vie_device_status.  Errors: VIE_ERR_INVALID_ARG, VIE_ERR_UNSUPPORTED,
 * VIE_ERR_CUDA.
 */
vie_status vie_head_topk_noalloc(const void *W_out, int64_t V, int32_t d, const float *h,
                                 int32_t batch, int32_t k, int32_t *out_idx, float *out_logits,
                                 vie_stream stream);

/*
 * vie_device_status - synchronises `stream`, then reads and clears the
 * library's device-side flag word of the current device.  Returns VIE_OK when
 * no kernel recorded a problem, VIE_ERR_DEVICE otherwise (vie_last_error()
 * names the problem), VIE_ERR_CUDA if the synchronisation itself failed.
 */
vie_status vie_device_status(vie_stream stream);

/* Same as vie_device_status for the handle's device, and also re-arms the
 * handle's scratch counters after a device-side problem. */
vie_status vie_head_device_status(vie_head *head, vie_stream stream);

/* Message for the last failing call on this thread ("" if none). */
const char *vie_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* VIE_HEAD_H */
