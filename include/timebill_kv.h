/*
 * timebill_kv.h - C ABI of the GB300 (sm_103a) KV-eviction + decode-attention
 * library behind TimeBill's eviction ratio alpha (arxiv 2512.21859).
 *
 * The paper chooses, per request, the fraction alpha of the prompt's KV cache
 * to evict after prefill (Eq. 14, Section "Time-Budgeted LLM Inference
 * Mechanism"), so that every decode step then attends over
 * N_kv = (1 - alpha) N_x + i - 1 keys (Eq. 8, Section "End-to-end Execution
 * Time Prediction"). It performs the eviction with SnapKV ("Experimental
 * Setup"). This library computes that eviction and the decode-step
 * attention over the compacted cache; choosing alpha stays with the caller.
 *
 * Conventions shared by every entry point
 * ----------------------------------------
 *  - The caller owns every buffer. Device buffers hold device addresses
 *    (allocated by the caller, e.g. with PyTorch); descriptor arrays marked
 *    "host" hold host addresses read during the call only. The library never
 *    allocates device memory; scratch comes from a caller-provided workspace
 *    whose size the *_workspace_size functions report.
 *  - Device calls are asynchronous on the given stream (NULL = the legacy
 *    default stream). Argument errors are returned synchronously, before
 *    anything is launched; the output buffers are then left untouched.
 *  - bf16 tensors are raw 16-bit bfloat16 values; f32 tensors IEEE float.
 *    Every device pointer must be 16-byte aligned.
 *  - No exceptions cross the ABI; every call returns a tb_status.
 *  - Calls that share a workspace must not overlap on the GPU.
 *  - The decode, select, gather and workspace-clearing kernels are launched
 *    with programmatic dependent launch: each may be scheduled while the
 *    kernel before it in the stream finishes, and waits for that kernel's
 *    completion before it touches global memory, so stream order holds as
 *    usual. Setting the environment variable TB_NO_PDL (read once per
 *    process) launches them the ordinary way.
 *
 * Notation: B requests; request b has prompt length N_b, eviction ratio
 * alpha_b and P_b = N_b - W prefix tokens (the last W prompt tokens form the
 * observation window). Hq query heads, Hkv KV heads, G = Hq / Hkv; query head
 * h reads KV head h / G. d = head_dim. k_b retained prefix tokens and
 * R_b = k_b + W retained rows per KV head (tb_retained_count).
 *
 * Packed layouts (row-major, innermost index last):
 *   q_win   [B][Hq][W][d]           window queries (the last W prompt rows)
 *   K, V    [Hkv][kv_rows][d]       request b at rows kv_offset[b] .. + N_b
 *   scores  [Hkv][score_rows] f32   request b at column sum_{b'<b} P_b'
 *   idx     [Hkv][idx_rows] int32   request b at column sum_{b'<b} R_b'
 *   Kc, Vc  [Hkv][out_rows][d]      request b at rows out_offset[b] .. + R_b
 *   score_rows = sum_b P_b, idx_rows = sum_b R_b (see tb_evict_layout).
 */
#ifndef TIMEBILL_KV_H
#define TIMEBILL_KV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream (cudaStream_t). */
typedef struct CUstream_st *tb_stream_t;

typedef enum {
  TB_OK = 0,
  TB_ERR_INVALID_ARG = 1,  /* null pointer, bad size, inconsistent layout */
  TB_ERR_UNSUPPORTED = 2,  /* valid but not built: head_dim, dtype, batch */
  TB_ERR_WORKSPACE = 3,    /* workspace missing, too small or misaligned */
  TB_ERR_CUDA = 4,         /* a CUDA launch or runtime call failed */
  TB_ERR_TIMEOUT = 5       /* a bounded device-side wait gave up */
} tb_status;

typedef enum { TB_F32 = 0, TB_BF16 = 1 } tb_dtype;

/* Largest batch one call accepts. */
#define TB_MAX_BATCH 64

/* Static description of a status code; never NULL. */
const char *tb_status_string(int32_t status);

/* Version of this ABI (major * 100 + minor): 103 (tb_decode_desc.max_ctas,
 * TB_DECODE_CONCURRENT, tb_select_ctas, TB_EVICT_GATHER_CONCURRENT). */
int32_t tb_abi_version(void);

/* Text of the last CUDA error this thread saw inside the library (the
 * cudaGetErrorString of the call behind a TB_ERR_CUDA), or "" if none. */
const char *tb_last_error_detail(void);

/* Kernels this library has launched in this process so far (all threads,
 * all devices). Lets a caller count the device work behind a region. */
uint64_t tb_launch_counter(void);

/*
 * Retained length (Eq. 8). k = ceil((1 - alpha) n - 1e-9 n) prefix tokens
 * survive on top of the W window tokens, clamped to [0, n - window]; the
 * 1e-9 n guard keeps a decimal alpha (0.3) from rounding up past an exact
 * product. Writes k to *k_out and k + window to *r_out.
 * Errors: TB_ERR_INVALID_ARG if a pointer is NULL, window < 1, n < window,
 * or alpha is outside [0, 1] (NaN included).
 */
tb_status tb_retained_count(int64_t n, int32_t window, double alpha,
                            int64_t *k_out, int64_t *r_out);

/* Bits of tb_evict_desc.flags (0 = the default readings). */
/* Eq. 8 read literally: the retained cache, window included, holds
 * ceil((1 - alpha) n) rows, so k = that count minus the window, clamped to
 * [0, n - window] (the window is still always kept). */
#define TB_EVICT_BUDGET_INCLUDES_WINDOW 1
/* Average pooling (SnapKV's own pooling) instead of max-pooling: pooled[j] =
 * (sum of the scores at [j - pool_k/2, j + pool_k/2] inside the prefix) /
 * pool_k, i.e. out-of-range neighbours count as zeros. */
#define TB_EVICT_AVG_POOL 2
/* For tb_gather_kv only (tb_score_evict ignores it: its gather waits for its
 * own select). The caller asserts that the kernel enqueued on the stream just
 * before the gather writes nothing the gather reads (idx, K, V), touches
 * neither Kc nor Vc, and that idx, K and V were complete before that kernel
 * was launched: the gather kernel then does not wait for that kernel before
 * its copies, so, launched behind one that lets its dependents start early,
 * it runs beside it (e.g. the gather of one layer beside the select of the
 * next). One of
 * its threads still waits for that kernel before it exits, so the gather
 * completes only after that kernel has: work ordered after the gather is
 * ordered after both. */
#define TB_EVICT_GATHER_CONCURRENT 4

/* tb_retained_count under the TB_EVICT_BUDGET_INCLUDES_WINDOW bit of
 * `flags` (other bits are ignored here). Same errors. */
tb_status tb_retained_count_ex(int64_t n, int32_t window, double alpha,
                               int32_t flags, int64_t *k_out, int64_t *r_out);

/* Shape of one batched eviction. All pointers are host arrays of length
 * `batch`, read during the call only. */
typedef struct {
  int32_t batch;     /* 1 .. TB_MAX_BATCH */
  int32_t hq;        /* query heads, a multiple of hkv */
  int32_t hkv;       /* KV heads */
  int32_t head_dim;  /* 64 or 128 */
  int32_t window;    /* observation window W >= 1 (W <= N_b) */
  int32_t pool_k;    /* max-pool kernel, odd, 1 .. 63 */
  int32_t dtype;     /* tb_dtype of q_win, K, V, Kc, Vc */
  int32_t flags;     /* TB_EVICT_* bits; any other bit is an error */
  const int64_t *n;          /* host [batch]: prompt lengths N_b */
  const double *alpha;       /* host [batch]: eviction ratios in [0, 1] */
  const int64_t *kv_offset;  /* host [batch]: first row of request b in K, V */
  int64_t kv_rows;           /* rows per KV head of K and V */
  const int64_t *out_offset; /* host [batch]: first row of request b in Kc, Vc */
  const int64_t *out_cap;    /* host [batch]: rows reserved for b (>= R_b) */
  int64_t out_rows;          /* rows per KV head of Kc and Vc */
} tb_evict_desc;

/*
 * Validates a descriptor and reports the packed sizes: *score_rows =
 * sum_b P_b and *idx_rows = sum_b R_b (either pointer may be NULL).
 * Errors: TB_ERR_INVALID_ARG (inconsistent descriptor, request rows outside
 * kv_rows / out_rows, out_cap < R_b), TB_ERR_UNSUPPORTED (head_dim, dtype).
 */
tb_status tb_evict_layout(const tb_evict_desc *desc, int64_t *score_rows,
                          int64_t *idx_rows);

/* Bytes of device workspace tb_window_scores, tb_select_topk and
 * tb_score_evict need for this descriptor (the same figure for all three). */
tb_status tb_evict_workspace_size(const tb_evict_desc *desc, size_t *bytes);

/*
 * Steps 1-3 of the eviction (SnapKV observation-window voting, named in
 * "Experimental Setup"; logits and softmax of the attention definition in
 * "FLOPs-based Modeling"): for every request, KV head g and prefix key j,
 *   scores[g][j] = sum over heads h of group g and window rows w of
 *                  softmax_j'( q_win[h][w] . K[g][j'] / sqrt(d) )[j],
 * where window row w sees keys j' <= P_b + w (causal). Writes `scores`
 * ([Hkv][score_rows] f32, device). Reads q_win, K (device).
 */
tb_status tb_window_scores(const tb_evict_desc *desc, const void *q_win,
                           const void *K, float *scores, void *workspace,
                           size_t workspace_bytes, tb_stream_t stream);

/*
 * tb_window_scores for a caller whose prefill attention already produced the
 * log-sum-exp of the observation-window rows (eviction runs right after the
 * prefill, Section "End-to-end Execution Time Prediction"; a flash-style
 * prefill kernel returns this per query row). With the row statistics
 * given, the scores need one Q K^T pass over the prefix keys instead of two:
 *   scores[g][j] = sum_{h in g, w < W} exp(q_win[h][w] . K[g][j] / sqrt(d)
 *                                          - lse[b][h][w]).
 * lse: device f32 [batch][Hq][W], 4-byte aligned: the natural log of
 * sum_{j' <= P_b + w} exp(q_win[h][w] . K[g][j'] / sqrt(d)) (the causal
 * window rows of tb_window_scores; with these values both calls give the
 * same scores up to rounding). Non-finite lse values give non-finite
 * scores; nothing checks them. Other arguments, outputs and errors as in
 * tb_window_scores; the workspace is the one tb_evict_workspace_size gives.
 */
tb_status tb_window_scores_lse(const tb_evict_desc *desc, const void *q_win,
                               const void *K, const float *lse, float *scores,
                               void *workspace, size_t workspace_bytes,
                               tb_stream_t stream);

/*
 * Steps 4-5: max-pool of the scores (kernel pool_k, stride 1, out-of-range
 * neighbours ignored), then per request and KV head the k_b prefix positions
 * with the largest pooled score (ties to the lower index) followed by the
 * window positions P_b .. N_b - 1, ascending, into idx ([Hkv][idx_rows]
 * int32, device; positions are relative to the request's first row).
 * `pooled` ([Hkv][score_rows] f32, device) receives the pooled scores, or
 * is NULL. Scores must be finite and >= 0.
 */
tb_status tb_select_topk(const tb_evict_desc *desc, const float *scores,
                         int32_t *idx, float *pooled, void *workspace,
                         size_t workspace_bytes, tb_stream_t stream);

/*
 * Number of CTAs the select of tb_select_topk (and of tb_score_evict) runs
 * for this descriptor, each on an SM of its own (a thread-block cluster of up
 * to eight per request and KV head; one per request and KV head on the
 * fallback path). A decode with TB_DECODE_CONCURRENT launched behind the
 * select fits beside it with max_ctas = SM count - this. No device work.
 */
tb_status tb_select_ctas(const tb_evict_desc *desc, int32_t *ctas);

/*
 * Step 6: Kc[g][out_offset[b] + r] = K[g][kv_offset[b] + idx[g][.. + r]]
 * and the same for V, for r < R_b (bit copies). idx entries must lie in
 * [0, N_b); an entry outside it is skipped and its row left untouched.
 */
tb_status tb_gather_kv(const tb_evict_desc *desc, const int32_t *idx,
                       const void *K, const void *V, void *Kc, void *Vc,
                       tb_stream_t stream);

/*
 * The whole eviction: tb_window_scores, tb_select_topk and tb_gather_kv in
 * one call (scores kept in the workspace). `pooled` may be NULL.
 */
tb_status tb_score_evict(const tb_evict_desc *desc, const void *q_win,
                         const void *K, const void *V, int32_t *idx,
                         void *Kc, void *Vc, float *pooled, void *workspace,
                         size_t workspace_bytes, tb_stream_t stream);

/* Bits of tb_decode_desc.flags. */
/* The caller asserts that the work enqueued on the stream just before a
 * tb_decode_attn_prepared call writes no row of Kc or Vc below lens[b] - 1
 * (the row a decode loop appends last, lens[b] - 1, may be written by it;
 * the rows before it were written earlier), and, if that work is a kernel
 * using programmatic dependent launch, that it lets its successor start
 * only after its own dependency wait. The decode kernel then requests its
 * first K/V tiles before that work has completed (hiding their latency
 * behind its tail) and reads row lens[b] - 1 again after it. No effect on
 * tb_decode_attn and tb_decode_attn_noalloc, whose own clearing kernel
 * already lets them do so. */
#define TB_DECODE_EARLY_CACHE_READ 1
/* The caller asserts that the work enqueued on the stream just before a
 * tb_decode_attn_prepared call writes nothing the call reads (q, Kc, Vc,
 * lens) and touches neither out nor the workspace, and that everything the
 * call reads was complete before that work was launched. The decode kernel
 * then does not wait for that work before its own: launched behind a kernel that
 * lets its dependents start early (the library's select and gather kernels
 * do, right after their own dependency wait), it runs beside it on the SMs
 * that kernel leaves free (size it with max_ctas, e.g. the SM count minus
 * tb_select_ctas). One of its threads still waits for the preceding
 * kernel before it exits, so the call completes only after that kernel
 * has: work ordered after the call is ordered after both. Implies
 * TB_DECODE_EARLY_CACHE_READ. No effect on tb_decode_attn and
 * tb_decode_attn_noalloc (their clearing kernel comes first). */
#define TB_DECODE_CONCURRENT 2

/* Shape of one batched decode step. */
typedef struct {
  int32_t batch;     /* 1 .. TB_MAX_BATCH */
  int32_t hq;        /* query heads, a multiple of hkv */
  int32_t hkv;       /* KV heads */
  int32_t head_dim;  /* 64 or 128 */
  int32_t dtype;     /* tb_dtype of q, Kc, Vc */
  int32_t out_dtype; /* tb_dtype of out: TB_F32, or equal to dtype */
  const int64_t *cache_offset; /* host [batch]: first row of b in Kc, Vc */
  const int64_t *cache_cap;    /* host [batch]: rows reserved for b */
  int64_t cache_rows;          /* rows per KV head of Kc and Vc */
  int64_t max_len;             /* upper bound of lens[b], >= 1 */
  int32_t flags;               /* TB_DECODE_* bits; any other bit is an error */
  int32_t max_ctas;            /* 0: about one CTA per SM of a 152-SM GB300
                                  (the keys of each (request, KV head) split
                                  that many ways); > 0: at most max(this,
                                  batch * hkv) CTAs, in fewer, longer splits;
                                  < 0 is an error */
} tb_decode_desc;

/* Bytes of device workspace tb_decode_attn needs for this descriptor. */
tb_status tb_decode_workspace_size(const tb_decode_desc *desc, size_t *bytes);

/*
 * One decode step (attention definition of "FLOPs-based Modeling" with a
 * single query row; N_kv^i keys per Eq. 8): for request b and query head h,
 *   out[b][h] = sum_{r < lens[b]} softmax_r(q[b][h] . Kc[g][r] / sqrt(d)) Vc[g][r]
 * with g = h / G and rows taken from request b's slice of Kc, Vc. The caller
 * appends the step's own K/V row at lens[b] - 1 beforehand.
 * q: [B][Hq][d] (dtype); out: [B][Hq][d] (out_dtype); lens: device int32 [B].
 * A length above min(max_len, cache_cap[b]) is clamped to it and flagged in
 * the workspace status word (tb_read_status); lens[b] <= 0 writes zeros.
 */
tb_status tb_decode_attn(const tb_decode_desc *desc, const void *q,
                         const void *Kc, const void *Vc, const int32_t *lens,
                         void *out, void *workspace, size_t workspace_bytes,
                         tb_stream_t stream);

/*
 * tb_decode_attn for a decode loop that keeps its workspace from step to
 * step (the paper has no counterpart: a deployment fast path). tb_decode_attn
 * zeroes the workspace's control words (status word, split counters) with a
 * small kernel before every step, which on GB300 costs about 1 us per call
 * between the previous kernel and this one; this entry point launches only
 * the decode kernel.
 *  - tb_decode_workspace_prepare zeroes the control words of a workspace of
 *    at least tb_decode_workspace_size bytes for `desc`; call it once after
 *    allocating the workspace (and again after any error or status flag).
 *    A workspace prepared for one descriptor serves every descriptor whose
 *    tb_decode_workspace_size is no larger and whose batch and hkv are the
 *    same (the split counters are indexed by request and KV head).
 *  - tb_decode_attn_prepared computes exactly what tb_decode_attn computes,
 *    with the same arguments; each call leaves the split counters at zero
 *    when it completes. The status word is not cleared between calls: a
 *    flag (a length above its cap, a bounded wait that gave up) stays set
 *    until the workspace is prepared again.
 *  - Calls sharing one workspace must not overlap on the GPU (one stream, or
 *    ordered by events), as for tb_decode_attn.
 * Errors: as tb_decode_attn.
 */
tb_status tb_decode_workspace_prepare(const tb_decode_desc *desc,
                                      void *workspace, size_t workspace_bytes,
                                      tb_stream_t stream);
tb_status tb_decode_attn_prepared(const tb_decode_desc *desc, const void *q,
                                  const void *Kc, const void *Vc,
                                  const int32_t *lens, void *out,
                                  void *workspace, size_t workspace_bytes,
                                  tb_stream_t stream);

/*
 * Waits for `stream`, then reads the status word kept at the start of a
 * workspace used by the calls above: TB_OK, TB_ERR_TIMEOUT (a bounded
 * device-side wait gave up) or TB_ERR_INVALID_ARG (a device-side range check
 * fired, e.g. a decode length above its cap). *raw (if not NULL) receives the
 * word itself. The word is cleared at the start of every call that can set
 * it: tb_window_scores, tb_score_evict and tb_decode_attn (tb_select_topk
 * never clears it and leaves it as it was; tb_gather_kv has no workspace;
 * tb_decode_attn_prepared keeps it until tb_decode_workspace_prepare).
 *
 * Debug build. libtimebill_kv_debug.so (the same entry points, built with
 * TB_DEBUG=1) also checks, on the device, invariants the release kernels
 * take for granted, and raises the same range bit (TB_ERR_INVALID_ARG here)
 * when one fails instead of trapping: every window row's log-sum-exp is
 * finite (non-finite inputs in q_win or K), tb_select_topk keeps exactly k
 * positions, tb_score_evict's gather sees only indices in [0, N_b), and a
 * decode head with keys has a positive finite softmax sum. The release
 * library compiles these checks out.
 */
tb_status tb_read_status(const void *workspace, size_t workspace_bytes,
                         tb_stream_t stream, int32_t *raw);

/*
 * Diagnostic of the bounded device-side waits behind TB_ERR_TIMEOUT
 * (failure detection; the paper has no counterpart). Every kernel here
 * waits on its barriers with a time limit and, when it runs out, raises the
 * workspace status word, waits for its own copies in flight, frees its
 * tensor memory and returns instead of hanging. This call runs that exit on
 * purpose: one CTA starts a 4 KB copy into shared memory, then waits on a
 * barrier that nothing completes (arrive = 0) for limit_ns nanoseconds of
 * the GPU timer, or on one it completes itself first (arrive = 1).
 *  - workspace: device, 256-byte aligned, at least 256 + 4096 bytes; its
 *    status word is cleared first, the 4 KB after the first 256 bytes are
 *    read (any contents). Afterwards tb_read_status on it gives
 *    TB_ERR_TIMEOUT (arrive = 0) or TB_OK (arrive = 1).
 *  - limit_ns: 10,000 .. 1,000,000,000 (10 us .. 1 s).
 * Errors: TB_ERR_WORKSPACE (missing, small or misaligned workspace),
 * TB_ERR_INVALID_ARG (limit out of range, arrive not 0 or 1), TB_ERR_CUDA.
 */
tb_status tb_diag_bounded_wait(void *workspace, size_t workspace_bytes,
                               uint64_t limit_ns, int32_t arrive,
                               tb_stream_t stream);

/* Size of the device array tb_decode_attn_noalloc uses as its scratch. */
#define TB_NOALLOC_SCRATCH_BYTES (4u << 20)

/*
 * tb_decode_attn for callers that cannot allocate device memory (the paper
 * has no counterpart: this is a deployment convenience). Some callers may not
 * call an allocator on their per-token path: a hard-real-time loop whose
 * deadline cannot absorb a cudaMalloc that may synchronise the device, or a
 * plugin inside a host framework that owns all device memory. This entry
 * point computes exactly what tb_decode_attn computes, with the same
 * arguments minus the workspace: its scratch is one library-owned device
 * array of TB_NOALLOC_SCRATCH_BYTES (4 MiB) that every GPU loading this
 * library holds until the process exits. It allocates nothing.
 *  - A descriptor whose tb_decode_workspace_size exceeds the array returns
 *    TB_ERR_WORKSPACE before any launch; use tb_decode_attn instead.
 *  - It runs on the calling thread's current device. The first call in each
 *    CUDA context (per device; a context made after cudaDeviceReset, or a
 *    driver-API context of the caller's, counts as new) looks up the array's
 *    device address there (cudaGetSymbolAddress) and keeps it, so make that
 *    first call before any stream capture.
 *  - Every call on a device shares the one array, which keeps the previous
 *    call's contents: calls that overlap on the GPU (other streams, other
 *    threads) race and must be serialised by the caller. Each call clears
 *    the array's status word and split counters before its kernels run.
 *  - A length above its cap is clamped and flagged as in tb_decode_attn,
 *    and a bounded wait that gives up raises the timeout flag (the output
 *    is then not valid); both flags land in the array's status word, which
 *    tb_decode_noalloc_status reads back.
 */
tb_status tb_decode_attn_noalloc(const tb_decode_desc *desc, const void *q,
                                 const void *Kc, const void *Vc,
                                 const int32_t *lens, void *out,
                                 tb_stream_t stream);

/*
 * Status word of the array tb_decode_attn_noalloc uses, on the current
 * device: waits for `stream` (the stream of the calls to check), then reports
 * what the last tb_decode_attn_noalloc call on this device raised, as
 * tb_read_status does: TB_OK, TB_ERR_TIMEOUT or TB_ERR_INVALID_ARG (a length
 * above its cap). *raw (if not NULL) receives the word. Allocates nothing.
 * Errors: TB_ERR_CUDA if the synchronisation or the read fails.
 */
tb_status tb_decode_noalloc_status(tb_stream_t stream, int32_t *raw);

/*
 * Execution-time model of "Profiling-based Fitting" (Eq. 6a and 6b), in
 * seconds: the prefill of N_x prompt tokens takes a N_x^2 + b N_x + c, one
 * decoding step over N_kv cached tokens takes p N_kv + q. Host memory.
 */
typedef struct {
  double a, b, c;
  double p, q;
} tb_time_model;

/*
 * Eq. 12: the worst-case execution time estimate of one request, in seconds:
 * the prefill of n_x tokens plus the decoding steps i = 1 .. n_w - 1, step i
 * over (1 - alpha) n_x + i - 1 cached tokens (Eqs. 9-11). n_w is the
 * pessimistic response length (tb_alpha_star reports the one it uses). Host
 * only; no device work.
 * Errors: TB_ERR_INVALID_ARG for a NULL pointer, n_x < 1, n_w < 1, alpha
 * outside [0, 1] or a non-finite coefficient.
 */
tb_status tb_wcet(const tb_time_model *model, int64_t n_x, double alpha,
                  int64_t n_w, double *t_out);

/*
 * The eviction ratio a time budget allows (Prob. 13 of "Time-Budgeted LLM
 * Inference Mechanism", closed form Eq. 14): the smallest alpha in
 * [0, alpha_max] with t_predict + WCET(alpha) <= budget, assuming the
 * pessimistic response length N_W = min(ceil(k * n_hat), n_max) (at least 1)
 * from the predicted length n_hat and the pessimistic factor k. When no alpha
 * in the range fits, alpha_max (the caller's overrun policy takes over).
 * In closed form, with n = N_W - 1 decoding steps:
 *   alpha = 1 - (budget - t_prefill - t_predict) / (p N_x n)
 *             + (n - 1) / (2 N_x) + q / (p N_x),   clamped to [0, alpha_max].
 * (The sum of Eq. 11 gives the middle term without p; the paper prints it
 * over 2 p N_x. The lower clamp is the alpha >= 0 constraint of Prob. 13.)
 * Writes *alpha_out and, if n_w_out is not NULL, N_W. Host only.
 * Errors: TB_ERR_INVALID_ARG for a NULL model or alpha_out, n_x < 1,
 * n_max < 1, n_hat < 0, k < 1, alpha_max outside [0, 1), p <= 0 or a
 * non-finite input.
 */
tb_status tb_alpha_star(const tb_time_model *model, int64_t n_x, double n_hat,
                        double k, int64_t n_max, double t_predict,
                        double budget, double alpha_max, double *alpha_out,
                        int64_t *n_w_out);

/*
 * Profiling-based fitting (Section "Profiling-based Fitting" of the
 * workload-guided execution time estimator): the least-squares polynomial
 * through measured (x_i, t_i) pairs, in the form of Eq. 6a (degree 2:
 * t = a x^2 + b x + c, x = N_x) or Eq. 6b (degree 1: t = p x + q,
 * x = N_kv). Host memory, host only; no device work.
 *  - x, t: count values each (any order, any units; t > 0).
 *  - coef_out: degree + 1 coefficients, highest power first ({a, b, c} or
 *    {p, q}), minimising sum_i (poly(x_i) - t_i)^2. Solved by Householder
 *    QR on the Vandermonde columns of x / max|x| (fp64), not by the normal
 *    equations, so N_x^2 ~ 1e9 costs no accuracy.
 *  - mape_out (may be NULL): the fit's mean absolute percentage error over
 *    the same points, 100 / count * sum_i |poly(x_i) - t_i| / t_i.
 * Errors: TB_ERR_INVALID_ARG for a NULL x, t or coef_out, degree other than
 * 1 or 2, fewer than degree + 1 distinct x values, a non-finite x or t, or
 * some t <= 0.
 */
tb_status tb_fit_time_model(const double *x, const double *t, int64_t count,
                            int32_t degree, double *coef_out,
                            double *mape_out);

#ifdef __cplusplus
}
#endif

#endif /* TIMEBILL_KV_H */
