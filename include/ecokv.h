/*
 * ecokv.h - C ABI of libecokv.so, the GB300 (sm_103a) ECOKV prefill
 * KV-cache eviction pass: score -> select -> compact.
 *
 * The method (ECOKV, "Geometry-Aware KV Cache Eviction via Complementary
 * Diversity Metrics"): for every layer l and KV head h, each cached key-value
 * pair i gets a score
 *
 *     S(i) = lambda * Stilde_div(i) + (1 - lambda) * S_imp(i)          (Eq. 7)
 *
 * where S_imp is the observation-window attention importance (SnapKV voting,
 * Appendix A), Stilde_div the rescaled composite Euclidean/cosine diversity
 * (Eq. 1-3 and the rescale of Sec. 5.2) and lambda the head-adaptive
 * redundancy weight (Eq. 4-6).  The top (budget - window) non-window pairs by
 * S are kept together with the whole observation window (Sec. 3 problem
 * statement), and the kept K/V rows are gathered into a compact cache.
 *
 * Conventions for every entry point
 * ---------------------------------
 *  - All tensor pointers are DEVICE pointers owned by the caller; the library
 *    never allocates device memory.  Scratch space is a caller-provided
 *    workspace of at least ecokv_workspace_size() bytes.
 *  - Layouts are dense row-major with d contiguous:
 *        K, V    [n_layers][h_kv][n][d]        (dtype)
 *        Qwin    [n_layers][h_q][window][d]    (dtype); row j of the window
 *                 is the query at position n - window + j
 *        S       [n_layers][h_kv][n - window]  float32 scores of the
 *                 non-window candidates
 *        lambda  [n_layers][h_kv]              float32
 *        idx     [n_layers][h_kv][n_keep]      int32, n_keep = min(budget, n):
 *                 the chosen candidates in ascending position, then the
 *                 window positions n - window .. n - 1
 *        K_out, V_out [n_layers][h_kv][n_keep][d] (dtype)
 *  - Query head q belongs to KV head q / (h_q / h_kv).
 *  - Pointers must be 16-byte aligned.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Argument errors are detected on the host and returned
 *    before anything is launched.  Errors found on the device (an index out of
 *    range handed to ecokv_compact, a bounded wait that gave up) are recorded
 *    in the workspace's status word; read them with ecokv_device_status().
 *  - Calls that share a workspace must be ordered on one stream.
 *  - Inputs must be finite; scores of non-finite inputs are unspecified.
 *  - Paths: bf16 inputs with n >= 128 stream K through a persistent
 *    tensor-core kernel, one launch for both of its passes over K, or one
 *    launch per group of at most 120 window rows when (h_q / h_kv) * window
 *    exceeds 120 (each group reads K twice); fp32 inputs, shorter caches and
 *    ECOKV_FLAG_FORCE_SIMT take the CUDA-core passes.  Every path is
 *    deterministic; scores may differ in their last bits between paths and
 *    between streaming schedules (ecokv_params.sched_*), within the
 *    documented tolerances.
 */
#ifndef ECOKV_H
#define ECOKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ECOKV_OK = 0,
  ECOKV_ERR_INVALID_ARG = 1,  /* bad sizes, null or misaligned pointers      */
  ECOKV_ERR_UNSUPPORTED = 2,  /* valid request this build does not handle     */
  ECOKV_ERR_WORKSPACE = 3,    /* workspace missing or smaller than required   */
  ECOKV_ERR_CUDA = 4,         /* a CUDA runtime call failed                   */
  ECOKV_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up           */
  ECOKV_ERR_DEVICE_INDEX = 6  /* device saw an index outside [0, n)           */
} ecokv_status;

typedef enum { ECOKV_F32 = 0, ECOKV_BF16 = 1 } ecokv_dtype;

/* variant flags (ecokv_params.flags) */
#define ECOKV_FLAG_SC_MIXKV_SIGN   0x1u /* s_C = -khat.mu (MixKV, Appendix A) instead of (1 - khat.mu)/2 */
#define ECOKV_FLAG_LAMBDA_OVERRIDE 0x2u /* use lambda_override for every head (0 = SnapKV importance only) */
#define ECOKV_FLAG_VNORM_IMP       0x4u /* S_imp(i) = pooled vote(i) * ||v_i||_2 (Sec. 5.2 combines the value
                                            norm with the window attention; the form is a reading).  Needs V:
                                            the ecokv_evict* entry points; ecokv_score returns
                                            ECOKV_ERR_UNSUPPORTED.  Heads of up to 131072 candidates
                                            (n - window), else ECOKV_ERR_UNSUPPORTED. */
#define ECOKV_FLAG_CENTROID_NONWIN 0x8u /* the centroid kbar of Eq. 1 over the n - window candidates only
                                            (Appendix B's alternative to Algorithm 1 step 5; all keys when
                                            n = window); d_E, D_E, mu and r_C otherwise as by default */
#define ECOKV_FLAG_WINSOR_1        0x10u /* winsorised min-max of Eq. 2: d_E clipped to its order statistics
                                             floor(p (n - W - 1)) and ceil((1 - p)(n - W - 1)) (0-based, no
                                             interpolation), p = 1 % (Appendix B's normalisation ablation) */
#define ECOKV_FLAG_WINSOR_5        0x20u /* the same with p = 5 %; at most one of the two.  Both: heads of up
                                             to 131072 candidates, else ECOKV_ERR_UNSUPPORTED */
#define ECOKV_FLAG_MAD             0x40u /* MAD scaling in place of the min-max of Eq. 2 (the same ablation):
                                             s_E = logistic((d_E - med) / (MAD + eps)), med the median of d_E
                                             over the candidates and MAD the median of |d_E - med| (an even
                                             count's median is the mean of its two middle values).  Not with
                                             a WINSOR flag (ECOKV_ERR_INVALID_ARG); heads of up to 131072
                                             candidates, else ECOKV_ERR_UNSUPPORTED */
#define ECOKV_FLAG_FORCE_SIMT      0x100u /* run the CUDA-core passes even where the tensor-core kernel applies */
#define ECOKV_FLAG_TEST_STALL      0x80000000u /* fault injection for tests of the bounded waits: the statistics of
                                             the first unit (layer 0, KV head 0) are never complete, so pass 2
                                             of that unit waits until timeout_us runs out; the call then records
                                             ECOKV_ERR_TIMEOUT in the workspace's status word and its outputs
                                             are unspecified.  Tensor-core path only (bf16, n >= 128), else
                                             ECOKV_ERR_UNSUPPORTED */

typedef struct {
  int32_t n_layers;    /* L >= 1 layers in one call                              */
  int32_t h_kv;        /* KV heads per layer, >= 1                                */
  int32_t h_q;         /* query heads per layer, a multiple of h_kv               */
  int32_t n;           /* cached tokens N (Sec. 3: T), 1 <= n <= 2^24             */
  int32_t d;           /* head dimension; this build supports d = 128             */
  int32_t window;      /* observation window W (Sec. 5.3), 1 <= W <= min(n, budget);
                          (h_q / h_kv) * W <= 256                                  */
  int32_t budget;      /* B retained tokens per head, window included; B >= n keeps all */
  int32_t pool_kernel; /* odd average-pooling width (Appendix A.3: 5)              */
  float alpha;         /* Eq. 3 weight of the Euclidean diversity, in [0, 1] (0.8) */
  float beta;          /* Eq. 6 weight of the Euclidean redundancy, in [0, 1] (0.6) */
  float tau;           /* Eq. 5 temperature; <= 0 selects sqrt(d)                  */
  float eps;           /* Eq. 2 min-max stabiliser, > 0 (1e-6)                     */
  uint32_t flags;      /* ECOKV_FLAG_* bits                                        */
  float lambda_override; /* lambda for every head when ECOKV_FLAG_LAMBDA_OVERRIDE  */
  /* Schedule of the streaming kernel (bf16 tensor-core path); 0 selects the
   * built-in default.  Results are deterministic for any setting, but the
   * grouping of floating-point partial sums follows the schedule (and the
   * device's SM count), so scores may differ in their last bits between
   * settings (within the tolerances).  ecokv_workspace_size depends on
   * sched_wave. */
  int32_t sched_wave;    /* heads (layer, KV head) per wave of the schedule (default: all heads, i.e. pass 1
                            of every head before any pass 2) */
  int32_t sched_lag;     /* waves between a wave's first and second read of its keys (default 1) */
  uint32_t timeout_us;   /* limit of every bounded device-side wait, microseconds (0 = 2 s); a wait that
                            runs out records ECOKV_ERR_TIMEOUT in the status word */
} ecokv_params;

/* Fill *p with the paper's defaults (Appendix A.3): alpha 0.8, beta 0.6,
 * tau sqrt(d), eps 1e-6, pool_kernel 5, window 4, flags 0, the default
 * schedule and wait limit.  Shape fields are zeroed and must be set by the
 * caller. */
void ecokv_params_default(ecokv_params* p);

/* Validate a parameter block.  Returns ECOKV_OK, ECOKV_ERR_INVALID_ARG (an
 * impossible request: W > n, B < W, even pool_kernel, h_q % h_kv != 0,
 * alpha/beta outside [0, 1], eps <= 0 ...) or ECOKV_ERR_UNSUPPORTED (d != 128,
 * (h_q/h_kv)*W > 256, n > 2^24). */
ecokv_status ecokv_check_params(const ecokv_params* p);

/* Bytes of device workspace the calls below need for *p (0 if *p is invalid).
 * The workspace holds per-chunk partial sums, per-head statistics, per-token
 * importance / distance / cosine arrays and the status word. */
size_t ecokv_workspace_size(const ecokv_params* p);

/* Scores of every non-window candidate (Eq. 1-7) and the per-head lambda.
 *   K, Qwin : inputs (dtype), see layouts above.
 *   S       : out, float32 [L][h_kv][n - W].
 *   lambda  : out, float32 [L][h_kv]; may be NULL.
 *   dbg     : out, optional (may be NULL), float32 [L][h_kv][5][n - W] holding,
 *             per candidate: raw window-attention sum, pooled importance S_imp,
 *             Euclidean distance d_E, cosine khat.mu and composite S_div. */
ecokv_status ecokv_score(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* Qwin,
                         float* S, float* lambda, float* dbg, void* ws, size_t ws_bytes, void* stream);

/* Per-head top-(B - W) selection over S (Sec. 3; ties go to the lower
 * position) followed by the window: idx [L][h_kv][min(B, n)] int32.  Exact
 * for any float32 S (radix select on the order-preserving integer image).
 * ws may be NULL (no device status). */
ecokv_status ecokv_select(const ecokv_params* p, const float* S, int32_t* idx, void* ws, size_t ws_bytes,
                          void* stream);

/* Gather the retained rows: K_out[l][h][r] = K[l][h][idx[l][h][r]], same for V.
 * Bit-exact copies.  An idx entry outside [0, n) yields a zero row and, when
 * ws is given, ECOKV_ERR_DEVICE_INDEX in the status word.  ws may be NULL. */
ecokv_status ecokv_compact(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                           const int32_t* idx, void* K_out, void* V_out, void* ws, size_t ws_bytes,
                           void* stream);

/* The whole pass: score, select and compact in one call.  S and lambda are
 * optional outputs (NULL to skip).  idx, K_out, V_out as above. */
ecokv_status ecokv_evict(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                         const void* Qwin, int32_t* idx, void* K_out, void* V_out, float* S,
                         float* lambda, void* ws, size_t ws_bytes, void* stream);

/* The whole pass with a budget per layer (PyramidKV, Appendix A): the heads
 * of layer l keep layer_budget[l] rows (window included; layer_budget[l] >= n
 * keeps the layer whole) instead of p->budget.
 *   layer_budget : host array of n_layers entries, each in [window, p->budget];
 *                  ecokv_pyramid_budgets gives PyramidKV's schedule.
 *   idx, K_out, V_out : as for ecokv_evict, with p->budget the per-head stride:
 *                  head (l, h) fills its first min(layer_budget[l], n) slots;
 *                  the idx slots after them hold -1 and those K_out / V_out
 *                  rows are not written.
 *   Everything else as for ecokv_evict.  n_layers <= 256 (else
 *   ECOKV_ERR_UNSUPPORTED). */
ecokv_status ecokv_evict_layered(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                 const void* Qwin, const int32_t* layer_budget, int32_t* idx, void* K_out,
                                 void* V_out, float* S, float* lambda, void* ws, size_t ws_bytes, void* stream);

/* PyramidKV's per-layer budgets (Appendix A) for n_layers layers keeping
 * n_layers * budget rows per head in all: b^{m-1} = total / (beta m),
 * b^0 = 2 total / m - b^{m-1}, linear in between, each rounded half up and at
 * least `window`.  beta > 0 shapes the pyramid (1 = uniform).  Host only. */
ecokv_status ecokv_pyramid_budgets(int32_t n_layers, int32_t budget, int32_t window, float beta, int32_t* out);

/* The whole pass with a layer-wide budget (AdaKV, Appendix A): instead of
 * each head keeping its own top-(B - W), the heads of a layer share one
 * budget of h_kv (B - W) candidates, taken as one top-K over their
 * concatenated scores (ties to the lower head, then the lower position); each
 * head keeps its window as well, so every layer keeps h_kv min(B, n) rows in
 * all, split unevenly between its heads.
 *   K, V, Qwin : as for ecokv_evict.
 *   idx        : out, int32 [L][h_kv * min(B, n)]: per layer the heads' lists
 *                in head order, each its kept candidates in ascending
 *                position, then its window N - W .. N - 1.
 *   head_off   : out, int32 [L][h_kv + 1]: head h's list is
 *                idx[l][head_off[l][h] .. head_off[l][h + 1]).
 *   K_out, V_out : out, [L][h_kv * min(B, n)][d], the rows idx names, in its order.
 *   lambda     : out, float32 [L][h_kv]; may be NULL.
 *   ws         : as for ecokv_evict (the same size).
 * B >= n keeps every row (head_off[l][h] = h n). */
ecokv_status ecokv_evict_adaptive(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                  const void* Qwin, int32_t* idx, int32_t* head_off, void* K_out,
                                  void* V_out, float* lambda, void* ws, size_t ws_bytes, void* stream);

/* ecokv_evict without a caller workspace and without any allocation.  The
 * paper has no counterpart: this is a deployment variant of the same pass for
 * callers that may not allocate device memory where they evict (a runtime
 * that gave all free HBM to its KV-cache pool, or C code with no allocator).
 *
 * The workspace is a fixed scratch area of ECOKV_NOALLOC_SCRATCH_BYTES
 * compiled into the library, one copy per device context, loaded with the
 * library's module on first use.  Nothing is allocated by the call: no
 * cudaMalloc, no allocating library routine.
 *   Arguments as for ecokv_evict, minus ws / ws_bytes, plus
 *   dev_status : optional device pointer, 4-byte aligned; in stream order
 *                after the pass it receives the call's device-side status (0,
 *                ECOKV_ERR_TIMEOUT or ECOKV_ERR_DEVICE_INDEX).  The scratch's
 *                status word is cleared at the end of every call, so with
 *                dev_status NULL a device-side error of the call is discarded
 *                and nothing reports it (ecokv_device_status cannot reach the
 *                scratch); pass a pointer wherever such errors matter.
 * Errors: everything ecokv_evict returns; ECOKV_ERR_WORKSPACE when the
 * workspace *p needs (ecokv_workspace_size) exceeds
 * ECOKV_NOALLOC_SCRATCH_BYTES, checked before anything is launched;
 * ECOKV_ERR_CUDA when the scratch's address cannot be obtained.
 * Set-up: the first call on a device looks the scratch's address up (with
 * that device current); make that first call before any stream capture.
 * Concurrency: all calls on one device share the scratch.  Calls whose
 * executions may overlap (unordered streams, several host threads) race on
 * it; issue them in one stream order. */
#define ECOKV_NOALLOC_SCRATCH_BYTES (16u << 20)
ecokv_status ecokv_evict_noalloc(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                                 const void* Qwin, int32_t* idx, void* K_out, void* V_out, float* S,
                                 float* lambda, uint32_t* dev_status, void* stream);

/* The whole pass for a KV cache resident in host memory.  The paper has no
 * counterpart: this is a deployment variant of ecokv_evict for caches kept in
 * host memory that the GPU can address (e.g. offloaded layers on a
 * Grace-Blackwell node), where the host link, not the GPU, sets the pace.
 *
 * Every host buffer below must be device-accessible at the same address:
 * pinned with cudaHostAlloc / cudaMallocHost, or registered with
 * cudaHostRegister(..., cudaHostRegisterMapped), on a system with unified
 * addressing.  Checked with cudaPointerGetAttributes before anything is
 * launched (ECOKV_ERR_INVALID_ARG otherwise).
 *   K, V, Qwin     : host inputs (dtype), layouts as for ecokv_evict.
 *   idx            : host out, int32 [L][h_kv][min(B, n)].
 *   K_out, V_out   : host out, [L][h_kv][min(B, n)][d].
 *   lambda         : host out, float32 [L][h_kv]; may be NULL.
 *   ws, ws_bytes   : device workspace of at least ecokv_workspace_size_host()
 *                    bytes, 16-byte aligned; it also holds the device copy of
 *                    K and Qwin and the indices.
 * Data movement, in stream order: K and Qwin are copied to the workspace once
 * (both streaming passes read them there); the gather reads the kept V rows
 * and writes K_out / V_out directly in host memory, so V crosses the host
 * link only for the kept rows; idx is copied back at the end.  Per call the
 * host link carries |K| + |Qwin| + B/n of |V| inbound and |K_out| + |V_out| +
 * |idx| outbound, against |K| + |V| + |Qwin| inbound for ecokv_evict on
 * copied inputs.  Exception: with ECOKV_FLAG_VNORM_IMP the value norms are
 * read from every row of V in host memory, so all of V crosses the link
 * once more (|K| + |V| + |Qwin| + B/n of |V| inbound).  Returns after enqueueing; the outputs are valid once
 * `stream` has reached that point.  Scores are not returned (use
 * ecokv_score on device copies for them). */
size_t ecokv_workspace_size_host(const ecokv_params* p, ecokv_dtype dtype);
ecokv_status ecokv_evict_host(const ecokv_params* p, ecokv_dtype dtype, const void* K, const void* V,
                              const void* Qwin, int32_t* idx, void* K_out, void* V_out, float* lambda,
                              void* ws, size_t ws_bytes, void* stream);

/* Synchronise `stream`, then read and clear the workspace's device status
 * word.  Returns ECOKV_OK, ECOKV_ERR_DEVICE_INDEX, ECOKV_ERR_TIMEOUT, or
 * ECOKV_ERR_CUDA if the synchronisation itself failed. */
ecokv_status ecokv_device_status(void* ws, void* stream);

/* Timing hook for benchmarks and profiling (no counterpart in the paper).
 * events: NULL to switch the hook off, else 4 cudaEvent_t handles created and
 * owned by the caller (n must be 4).  While set, every ecokv_score /
 * ecokv_evict call made from this host thread records, on its stream,
 * events[0] before the streaming kernel(s), events[1] after them, events[2]
 * after the finalize / select kernel and (ecokv_evict only) events[3] after
 * the compaction kernel, so that cudaEventElapsedTime gives each stage's
 * device time.  Returns ECOKV_ERR_INVALID_ARG if events != NULL and n != 4. */
ecokv_status ecokv_set_stage_events(void* const* events, int n);

/* Static text for a status code. */
const char* ecokv_status_string(ecokv_status s);

#ifdef __cplusplus
}
#endif

#endif /* ECOKV_H */
