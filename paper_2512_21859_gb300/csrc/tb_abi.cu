// C-ABI entry points: argument validation, workspace carving, launch order.
//
// Every check runs on the host before the first CUDA call, so an invalid
// call returns without touching the GPU or any output buffer.
#include <cuda_runtime.h>

#include <cmath>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <vector>
#include <atomic>

#include <nvtx3/nvToolsExt.h>

#include "tb_internal.cuh"

namespace tb {

// A named NVTX range around a compute entry point (its host-side launch
// sequence), for timeline tools: ncu --nvtx, Nsight Systems. Without a tool
// attached a range costs a function-pointer check.
NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

namespace {

thread_local char g_last_error[256] = "";
std::atomic<uint64_t> g_launches{0};

}  // namespace

tb_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return TB_OK;
  strncpy(g_last_error, cudaGetErrorString(e), sizeof(g_last_error) - 1);
  g_last_error[sizeof(g_last_error) - 1] = '\0';
  return TB_ERR_CUDA;
}

namespace {

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// k = ceil((1 - alpha) n - 1e-9 n), clamped to [0, n - window] (Eq. 8 reading).
bool retained(int64_t n, int32_t window, double alpha, int32_t flags, int64_t* k, int64_t* r) {
  if (window < 1 || n < window) return false;
  if (!(alpha >= 0.0 && alpha <= 1.0)) return false;
  const double x = (1.0 - alpha) * (double)n - 1e-9 * (double)n;
  int64_t kk = (int64_t)ceil(x);
  if (flags & TB_EVICT_BUDGET_INCLUDES_WINDOW) kk -= window;
  const int64_t p = n - window;
  if (kk < 0) kk = 0;
  if (kk > p) kk = p;
  *k = kk;
  *r = kk + window;
  return true;
}

bool ranges_overlap(const int64_t* off, const int64_t* len, int batch) {
  for (int a = 0; a < batch; ++a)
    for (int b = a + 1; b < batch; ++b)
      if (len[a] > 0 && len[b] > 0 && off[a] < off[b] + len[b] && off[b] < off[a] + len[a])
        return true;
  return false;
}

tb_status build_evict(const tb_evict_desc* d, EvictParams* p) {
  if (!d) return TB_ERR_INVALID_ARG;
  if (d->batch < 1 || d->hq < 1 || d->hkv < 1 || d->window < 1 ||
      (d->flags & ~(TB_EVICT_BUDGET_INCLUDES_WINDOW | TB_EVICT_AVG_POOL |
                    TB_EVICT_GATHER_CONCURRENT)) != 0)
    return TB_ERR_INVALID_ARG;
  if (d->batch > TB_MAX_BATCH) return TB_ERR_UNSUPPORTED;
  if (d->hq % d->hkv != 0) return TB_ERR_INVALID_ARG;
  if (d->pool_k < 1 || d->pool_k % 2 == 0 || d->pool_k > 63) return TB_ERR_INVALID_ARG;
  if (d->dtype != TB_F32 && d->dtype != TB_BF16) return TB_ERR_UNSUPPORTED;
  if (d->head_dim != 64 && d->head_dim != 128) return TB_ERR_UNSUPPORTED;
  if (!d->n || !d->alpha || !d->kv_offset || !d->out_offset || !d->out_cap)
    return TB_ERR_INVALID_ARG;
  if (d->kv_rows < 0 || d->out_rows < 0) return TB_ERR_INVALID_ARG;
  const int group = d->hq / d->hkv;
  const int64_t m_rows = (int64_t)group * d->window;
  if (m_rows > kMaxWindowRows) return TB_ERR_UNSUPPORTED;

  memset(p, 0, sizeof(*p));
  p->batch = d->batch;
  p->hq = d->hq;
  p->hkv = d->hkv;
  p->group = group;
  p->d = d->head_dim;
  p->window = d->window;
  p->pool_k = d->pool_k;
  p->flags = d->flags;
  p->dtype = d->dtype;
  p->m_rows = (int32_t)m_rows;
  p->chunk = kSimtChunk;
  p->kv_rows = d->kv_rows;
  p->out_rows = d->out_rows;
  p->scale_log2 = (float)(1.4426950408889634 / sqrt((double)d->head_dim));
  p->rowc_scale = 1.0f;

  int64_t score_rows = 0, idx_rows = 0, items = 0;
  int64_t rlen[TB_MAX_BATCH];
  for (int b = 0; b < d->batch; ++b) {
    const int64_t n = d->n[b];
    if (n < d->window || n > (int64_t(1) << 30)) return TB_ERR_INVALID_ARG;
    int64_t k, r;
    if (!retained(n, d->window, d->alpha[b], d->flags, &k, &r)) return TB_ERR_INVALID_ARG;
    if (d->kv_offset[b] < 0 || d->kv_offset[b] + n > d->kv_rows) return TB_ERR_INVALID_ARG;
    if (d->out_offset[b] < 0 || d->out_cap[b] < r ||
        d->out_offset[b] + d->out_cap[b] > d->out_rows)
      return TB_ERR_INVALID_ARG;
    EvictReq& q = p->req[b];
    q.kv_off = d->kv_offset[b];
    q.out_off = d->out_offset[b];
    q.score_off = score_rows;
    q.idx_off = idx_rows;
    q.n = (int32_t)n;
    q.p = (int32_t)(n - d->window);
    q.k = (int32_t)k;
    q.item0 = (int32_t)items;
    score_rows += n - d->window;
    idx_rows += r;
    items += (int64_t)d->hkv * ((n + p->chunk - 1) / p->chunk);
    if (items > (int64_t)0x7fffffff) return TB_ERR_UNSUPPORTED;
    p->max_p = std::max<int32_t>(p->max_p, q.p);
    p->max_r = std::max<int32_t>(p->max_r, (int32_t)r);
    rlen[b] = d->out_cap[b];
  }
  if (ranges_overlap(d->out_offset, rlen, d->batch)) return TB_ERR_INVALID_ARG;
  p->items = (int32_t)items;
  p->score_rows = score_rows;
  p->idx_rows = idx_rows;
  return TB_OK;
}

EvictWorkspace carve_evict(const EvictParams& p) {
  EvictWorkspace w;
  size_t off = 0;
  w.status = off;
  off += kStatusBytes;
  w.tilectr = off;
  off = align_up(off + 2 * sizeof(int32_t) * (size_t)p.batch * p.hkv, 256);
  w.lsum = off;
  off = align_up(off + sizeof(double) * (size_t)p.batch * p.hkv * p.m_rows, 256);
  w.zeroed = off;
  w.scores = off;
  off = align_up(off + sizeof(float) * (size_t)p.hkv * p.score_rows, 256);
  w.partial = off;
  off = align_up(off + sizeof(float2) * (size_t)p.items * p.m_rows, 256);
  w.rowc = off;
  off = align_up(off + sizeof(float) * (size_t)p.batch * p.hkv * p.m_rows, 256);
  w.pooled = off;
  off = align_up(off + sizeof(float) * (size_t)p.hkv * p.score_rows, 256);
  w.total = off;
  return w;
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

tb_status check_ws(void* ws, size_t bytes, size_t need) {
  if (!ws || bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return TB_ERR_WORKSPACE;
  return TB_OK;
}

}  // namespace

tb_status build_decode(const tb_decode_desc* d, DecodeParams* p) {
  if (!d) return TB_ERR_INVALID_ARG;
  if (d->batch < 1 || d->hq < 1 || d->hkv < 1 || d->max_len < 1) return TB_ERR_INVALID_ARG;
  if ((d->flags & ~(TB_DECODE_EARLY_CACHE_READ | TB_DECODE_CONCURRENT)) != 0 || d->max_ctas < 0)
    return TB_ERR_INVALID_ARG;
  if (d->batch > TB_MAX_BATCH) return TB_ERR_UNSUPPORTED;
  if (d->hq % d->hkv != 0) return TB_ERR_INVALID_ARG;
  if (d->dtype != TB_F32 && d->dtype != TB_BF16) return TB_ERR_UNSUPPORTED;
  if (d->out_dtype != TB_F32 && d->out_dtype != d->dtype) return TB_ERR_UNSUPPORTED;
  if (d->head_dim != 64 && d->head_dim != 128) return TB_ERR_UNSUPPORTED;
  if (!d->cache_offset || !d->cache_cap || d->cache_rows < 0) return TB_ERR_INVALID_ARG;
  if (d->max_len > (int64_t(1) << 30)) return TB_ERR_UNSUPPORTED;
  const int group = d->hq / d->hkv;
  const int hs = 128 / d->head_dim;
  if ((group + hs - 1) / hs > 32) return TB_ERR_UNSUPPORTED;
  memset(p, 0, sizeof(*p));
  p->batch = d->batch;
  p->hq = d->hq;
  p->hkv = d->hkv;
  p->group = group;
  p->d = d->head_dim;
  p->dtype = d->dtype;
  p->out_dtype = d->out_dtype;
  p->cache_rows = d->cache_rows;
  p->max_len = d->max_len;
  p->scale_log2 = (float)(1.4426950408889634 / sqrt((double)d->head_dim));
  for (int b = 0; b < d->batch; ++b) {
    if (d->cache_offset[b] < 0 || d->cache_cap[b] < 0 ||
        d->cache_offset[b] + d->cache_cap[b] > d->cache_rows)
      return TB_ERR_INVALID_ARG;
    if (d->cache_cap[b] > (int64_t(1) << 30)) return TB_ERR_UNSUPPORTED;
    p->cache_off[b] = d->cache_offset[b];
    p->cache_cap[b] = (int32_t)d->cache_cap[b];
  }
  // Split the keys so that about one CTA per SM of a 152-SM part runs, in
  // whole 128-key tiles (each CTA keeps three tiles in flight); with a CTA
  // budget, as many splits per (request, KV head) as it holds (at least one).
  // Rounding the split length up to whole tiles only lowers the count.
  const int64_t units = (int64_t)d->batch * d->hkv;
  int64_t splits = d->max_ctas > 0 ? d->max_ctas / units : (152 + units - 1) / units;
  const int64_t max_splits = (d->max_len + 127) / 128;
  splits = std::max<int64_t>(1, std::min(splits, max_splits));
  int64_t split_len = (d->max_len + splits - 1) / splits;
  split_len = (split_len + 127) / 128 * 128;
  splits = (d->max_len + split_len - 1) / split_len;
  p->splits = (int32_t)splits;
  p->split_len = (int32_t)split_len;
  p->early_tma = 1;
  // When every split is a single 128-key tile (short caches), a merge kernel
  // behind the split kernel merges the splits (four CTAs per KV head, each
  // on a quarter of the head dims); with longer splits the last split CTA of
  // each (request, KV head) does. Measured on GB300 (graphs of consecutive
  // prepared calls, µs, last CTA -> merge kernel): one-tile splits: 7B shape
  // at 2K keys 5.81 -> 5.23, at 4K 6.42 -> 5.92, 32K α 0.95 5.73 -> 5.15;
  // longer splits: 7B shape at 8K 7.65 -> 7.81, 32K α 0.75 7.64 -> 7.81,
  // α 0.5 10.23 -> 10.45, 128K α 0.75 25.69 -> 25.92, α 0.9 13.75 -> 13.59.
  p->merge_kernel = split_len <= 128 ? 1 : 0;
  return TB_OK;
}

DecodeWorkspace carve_decode(const DecodeParams& p) {
  DecodeWorkspace w;
  size_t off = 0;
  w.status = off;
  off += kStatusBytes;
  w.counters = off;
  off = align_up(off + sizeof(int32_t) * (size_t)p.batch * p.hkv, 256);
  w.part_o = off;
  off = align_up(off + sizeof(float) * (size_t)p.batch * p.hq * p.splits * p.d, 256);
  w.part_ml = off;
  off = align_up(off + sizeof(float2) * (size_t)p.batch * p.hq * p.splits, 256);
  w.total = off;
  return w;
}

namespace {

template <typename T>
T* at(void* base, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(base) + off);
}

// The control words every eviction call clears: the status area and the
// tile counters, and the fp64 row sums when the scoring kernel uses them.
size_t evict_clear_bytes(const EvictParams& p, const EvictWorkspace& w) {
  return window_scores_row_sums(p) ? w.zeroed : w.lsum;
}

tb_status run_window_scores(const EvictParams& p, const EvictWorkspace& w, const void* q_win,
                            const void* K, float* scores, void* ws, cudaStream_t s) {
  return cuda_status(launch_window_scores(p, q_win, K, scores, at<float2>(ws, w.partial),
                                          at<float>(ws, w.rowc), at<int32_t>(ws, w.status),
                                          at<int32_t>(ws, w.tilectr), at<double>(ws, w.lsum), s));
}

tb_status run_select(const EvictParams& p, const EvictWorkspace& w, const float* scores,
                     int32_t* idx, float* pooled, void* ws, cudaStream_t s) {
  int32_t* status = at<int32_t>(ws, w.status);
  if (select_cluster_supported(p))
    return cuda_status(launch_select_cluster(p, scores, pooled, idx, status, s));
  float* pl = pooled ? pooled : at<float>(ws, w.pooled);
  cudaError_t e = launch_pool(p, scores, pl, s);
  if (e == cudaSuccess) e = launch_select(p, pl, idx, status, s);
  return cuda_status(e);
}

}  // namespace

void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

bool pdl_enabled() {
  static const bool on = getenv("TB_NO_PDL") == nullptr;
  return on;
}

namespace {

// Clears a workspace's control words (status word, split / tile counters)
// ahead of the call's kernels. A kernel node costs about a fifth of what a
// memset node does inside a CUDA graph (~0.7 vs ~3.5 us between kernels).
__global__ void clear_words(uint4* __restrict__ w, size_t n16) {
  pdl_wait();
  pdl_trigger();
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16;
       i += (size_t)gridDim.x * blockDim.x)
    w[i] = make_uint4(0u, 0u, 0u, 0u);
}

// The same, and the nf floats at f (16-byte aligned) as well: the scores the
// votes-only scoring adds into, in the same launch.
__global__ void clear_words_and_floats(uint4* __restrict__ w, size_t n16, float* __restrict__ f,
                                       size_t nf) {
  pdl_wait();
  pdl_trigger();
  const size_t nf16 = nf / 4, total = n16 + nf16;
  uint4* f4 = reinterpret_cast<uint4*>(f);
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    if (i < n16) w[i] = make_uint4(0u, 0u, 0u, 0u);
    else f4[i - n16] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (blockIdx.x == 0 && threadIdx.x < (nf & 3)) f[nf16 * 4 + threadIdx.x] = 0.f;
}

cudaError_t clear_control_words_and_floats(void* ws, size_t bytes, float* f, size_t nf,
                                           cudaStream_t s) {
  const size_t n16 = bytes / 16;  // callers pass multiples of 256 bytes
  const size_t total = n16 + nf / 4 + 1;
  const unsigned blocks = (unsigned)std::min<size_t>((total + 255) / 256, 152);
  const cudaError_t e = launch_pdl(clear_words_and_floats, dim3(blocks), dim3(256), 0, s,
                                   static_cast<uint4*>(ws), n16, f, nf);
  count_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t clear_control_words(void* ws, size_t bytes, cudaStream_t s) {
  const size_t n16 = bytes / 16;  // callers pass multiples of 256 bytes
  if (n16 == 0) return cudaSuccess;
  const unsigned blocks = (unsigned)std::min<size_t>((n16 + 255) / 256, 152);
  const cudaError_t e =
      launch_pdl(clear_words, dim3(blocks), dim3(256), 0, s, static_cast<uint4*>(ws), n16);
  count_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_window_votes(const EvictParams& p, const void* q_win, const void* K,
                                float* scores, const float* rowc, int32_t* status,
                                int32_t* tilectr, cudaStream_t s) {
  if (window_scores_tc_supported(p))
    return launch_window_votes_tc(p, q_win, K, scores, rowc, status, tilectr, s);
  return launch_window_votes_simt(p, q_win, K, scores, rowc, s);
}

cudaError_t launch_window_scores(const EvictParams& p, const void* q_win, const void* K,
                                 float* scores, float2* partial, float* rowc, int32_t* status,
                                 int32_t* tilectr, double* lsum, cudaStream_t s) {
  if (window_scores_tc_supported(p))
    return launch_window_scores_tc(p, q_win, K, scores, partial, rowc, status, tilectr, lsum, s);
  return launch_window_scores_simt(p, q_win, K, scores, partial, rowc, s);
}

}  // namespace tb

using namespace tb;

extern "C" {

const char* tb_status_string(int32_t status) {
  switch (status) {
    case TB_OK: return "ok";
    case TB_ERR_INVALID_ARG: return "invalid argument";
    case TB_ERR_UNSUPPORTED: return "unsupported configuration";
    case TB_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case TB_ERR_CUDA: return "CUDA error";
    case TB_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
  }
}

int32_t tb_abi_version(void) { return 103; }

const char* tb_last_error_detail(void) { return g_last_error; }

uint64_t tb_launch_counter(void) { return g_launches.load(std::memory_order_relaxed); }

tb_status tb_retained_count(int64_t n, int32_t window, double alpha, int64_t* k_out,
                            int64_t* r_out) {
  return tb_retained_count_ex(n, window, alpha, 0, k_out, r_out);
}

tb_status tb_retained_count_ex(int64_t n, int32_t window, double alpha, int32_t flags,
                               int64_t* k_out, int64_t* r_out) {
  if (!k_out || !r_out) return TB_ERR_INVALID_ARG;
  int64_t k, r;
  if (!retained(n, window, alpha, flags, &k, &r)) return TB_ERR_INVALID_ARG;
  *k_out = k;
  *r_out = r;
  return TB_OK;
}

namespace {

bool model_ok(const tb_time_model* m) {
  return m && std::isfinite(m->a) && std::isfinite(m->b) && std::isfinite(m->c) &&
         std::isfinite(m->p) && std::isfinite(m->q);
}

double prefill_time(const tb_time_model* m, double nx) { return (m->a * nx + m->b) * nx + m->c; }

}  // namespace

// Eq. 12 with the decoding-phase sum of Eq. 11 in closed form:
// sum_{i=1..n} p((1 - alpha) N_x + i - 1) + q = n p (1 - alpha) N_x + p n (n - 1) / 2 + n q.
tb_status tb_wcet(const tb_time_model* model, int64_t n_x, double alpha, int64_t n_w,
                  double* t_out) {
  if (!model_ok(model) || !t_out || n_x < 1 || n_w < 1 || !(alpha >= 0.0 && alpha <= 1.0))
    return TB_ERR_INVALID_ARG;
  const double nx = (double)n_x, n = (double)(n_w - 1);
  *t_out = prefill_time(model, nx) + n * model->p * (1.0 - alpha) * nx +
           model->p * n * (n - 1.0) / 2.0 + n * model->q;
  return TB_OK;
}

// Prob. 13 through the closed form of Eq. 14 (with the middle term as the
// sum of Eq. 11 gives it, and the alpha >= 0 clamp): the constraint
// t_predict + WCET(alpha) <= budget is linear in alpha with slope -p N_x n.
tb_status tb_alpha_star(const tb_time_model* model, int64_t n_x, double n_hat, double k,
                        int64_t n_max, double t_predict, double budget, double alpha_max,
                        double* alpha_out, int64_t* n_w_out) {
  if (!model_ok(model) || !alpha_out || n_x < 1 || n_max < 1 || !(n_hat >= 0.0) ||
      !std::isfinite(n_hat) || !(k >= 1.0) || !std::isfinite(k) || !(model->p > 0.0) ||
      !(alpha_max >= 0.0 && alpha_max < 1.0) || !std::isfinite(t_predict) ||
      !std::isfinite(budget))
    return TB_ERR_INVALID_ARG;
  const double kn = std::ceil(k * n_hat);
  int64_t n_w = kn >= (double)n_max ? n_max : (int64_t)kn;
  if (n_w < 1) n_w = 1;
  const double nx = (double)n_x, n = (double)(n_w - 1);
  const double slack = budget - prefill_time(model, nx) - t_predict;
  double alpha;
  if (n_w == 1) {
    alpha = slack >= 0.0 ? 0.0 : alpha_max;  // no decoding step: alpha cannot help
  } else {
    const double req = 1.0 - slack / (model->p * nx * n) + (n - 1.0) / (2.0 * nx) +
                       model->q / (model->p * nx);
    alpha = std::fmin(alpha_max, std::fmax(0.0, req));
  }
  *alpha_out = alpha;
  if (n_w_out) *n_w_out = n_w;
  return TB_OK;
}

// Least squares of the profiling-based fit (Eq. 6a / 6b coefficients):
// Householder QR of the (count x (degree + 1)) Vandermonde matrix of the
// scaled abscissae u = x / s, then back substitution; the coefficient of u^k
// is divided by s^k at the end.
tb_status tb_fit_time_model(const double* x, const double* t, int64_t count, int32_t degree,
                            double* coef_out, double* mape_out) {
  if (!x || !t || !coef_out || (degree != 1 && degree != 2) || count < degree + 1)
    return TB_ERR_INVALID_ARG;
  double s = 0.0;
  for (int64_t i = 0; i < count; ++i) {
    if (!std::isfinite(x[i]) || !std::isfinite(t[i]) || !(t[i] > 0.0)) return TB_ERR_INVALID_ARG;
    s = std::fmax(s, std::fabs(x[i]));
  }
  {
    std::vector<double> xs(x, x + count);
    std::sort(xs.begin(), xs.end());
    if (std::unique(xs.begin(), xs.end()) - xs.begin() < degree + 1) return TB_ERR_INVALID_ARG;
  }
  if (s == 0.0) s = 1.0;
  const int nc = degree + 1;  // columns: u^degree, ..., u, 1
  const size_t n = (size_t)count;
  std::vector<double> A(n * nc), y(t, t + count);
  for (size_t i = 0; i < n; ++i) {
    const double u = x[i] / s;
    double pw = 1.0;
    for (int c = nc - 1; c >= 0; --c) {
      A[i * nc + c] = pw;
      pw *= u;
    }
  }
  std::vector<double> v(n);
  for (int c = 0; c < nc; ++c) {
    double norm = 0.0;
    for (size_t i = c; i < n; ++i) norm = std::hypot(norm, A[i * nc + c]);
    if (norm == 0.0) return TB_ERR_INVALID_ARG;
    const double alpha = A[c * nc + c] > 0.0 ? -norm : norm;
    double vn = 0.0;
    for (size_t i = c; i < n; ++i) {
      v[i] = A[i * nc + c] - (i == (size_t)c ? alpha : 0.0);
      vn += v[i] * v[i];
    }
    if (vn > 0.0) {
      for (int j = c; j < nc; ++j) {
        double d = 0.0;
        for (size_t i = c; i < n; ++i) d += v[i] * A[i * nc + j];
        d = 2.0 * d / vn;
        for (size_t i = c; i < n; ++i) A[i * nc + j] -= d * v[i];
      }
      double d = 0.0;
      for (size_t i = c; i < n; ++i) d += v[i] * y[i];
      d = 2.0 * d / vn;
      for (size_t i = c; i < n; ++i) y[i] -= d * v[i];
    }
  }
  double cu[3] = {0.0, 0.0, 0.0};
  for (int c = nc - 1; c >= 0; --c) {
    double r = y[c];
    for (int j = c + 1; j < nc; ++j) r -= A[c * nc + j] * cu[j];
    if (A[c * nc + c] == 0.0) return TB_ERR_INVALID_ARG;
    cu[c] = r / A[c * nc + c];
  }
  for (int c = 0; c < nc; ++c) coef_out[c] = cu[c] / std::pow(s, (double)(nc - 1 - c));
  if (mape_out) {
    double acc = 0.0;
    for (size_t i = 0; i < n; ++i) {
      double f = 0.0;
      for (int c = 0; c < nc; ++c) f = f * x[i] + coef_out[c];
      acc += std::fabs(f - t[i]) / t[i];
    }
    *mape_out = 100.0 * acc / (double)n;
  }
  return TB_OK;
}

tb_status tb_evict_layout(const tb_evict_desc* desc, int64_t* score_rows, int64_t* idx_rows) {
  EvictParams p;
  const tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (score_rows) *score_rows = p.score_rows;
  if (idx_rows) *idx_rows = p.idx_rows;
  return TB_OK;
}

tb_status tb_evict_workspace_size(const tb_evict_desc* desc, size_t* bytes) {
  if (!bytes) return TB_ERR_INVALID_ARG;
  EvictParams p;
  const tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  *bytes = carve_evict(p).total;
  return TB_OK;
}

tb_status tb_window_scores(const tb_evict_desc* desc, const void* q_win, const void* K,
                           float* scores, void* workspace, size_t workspace_bytes,
                           tb_stream_t stream) {
  const NvtxRange range("tb_window_scores");
  EvictParams p;
  tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (!q_win || !K || !scores || !aligned16(q_win) || !aligned16(K) || !aligned16(scores))
    return TB_ERR_INVALID_ARG;
  const EvictWorkspace w = carve_evict(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = cuda_status(clear_control_words(workspace, evict_clear_bytes(p, w), s))) != TB_OK) return st;
  return run_window_scores(p, w, q_win, K, scores, workspace, s);
}

tb_status tb_window_scores_lse(const tb_evict_desc* desc, const void* q_win, const void* K,
                               const float* lse, float* scores, void* workspace,
                               size_t workspace_bytes, tb_stream_t stream) {
  const NvtxRange range("tb_window_scores_lse");
  EvictParams p;
  tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (!q_win || !K || !lse || !scores || !aligned16(q_win) || !aligned16(K) ||
      !aligned16(scores) || (reinterpret_cast<uintptr_t>(lse) & 3u) != 0)
    return TB_ERR_INVALID_ARG;
  const EvictWorkspace w = carve_evict(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // the tensor-core votes kernel adds the quarters of each key's sum into the
  // scores, so it gets them cleared with the control words
  if (window_scores_tc_supported(p))
    st = cuda_status(clear_control_words_and_floats(workspace, evict_clear_bytes(p, w), scores,
                                                    (size_t)p.hkv * (size_t)p.score_rows, s));
  else
    st = cuda_status(clear_control_words(workspace, evict_clear_bytes(p, w), s));
  if (st != TB_OK) return st;
  p.rowc_scale = 1.4426950408889634f;  // natural-log LSE -> log2 units
  return cuda_status(launch_window_votes(p, q_win, K, scores, lse, at<int32_t>(workspace, w.status),
                                         at<int32_t>(workspace, w.tilectr), s));
}

tb_status tb_select_topk(const tb_evict_desc* desc, const float* scores, int32_t* idx,
                         float* pooled, void* workspace, size_t workspace_bytes,
                         tb_stream_t stream) {
  const NvtxRange range("tb_select_topk");
  EvictParams p;
  tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (!scores || !idx || !aligned16(scores) || !aligned16(idx) || (pooled && !aligned16(pooled)))
    return TB_ERR_INVALID_ARG;
  const EvictWorkspace w = carve_evict(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // the select kernels neither set the status word nor use the counters, so
  // the workspace is not cleared here (one graph node less per eviction)
  return run_select(p, w, scores, idx, pooled, workspace, s);
}

tb_status tb_select_ctas(const tb_evict_desc* desc, int32_t* ctas) {
  if (!ctas) return TB_ERR_INVALID_ARG;
  EvictParams p;
  const tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  const int per = select_cluster_supported(p) ? select_cluster_size(p) : 1;
  *ctas = p.batch * p.hkv * per;
  return TB_OK;
}

tb_status tb_gather_kv(const tb_evict_desc* desc, const int32_t* idx, const void* K,
                       const void* V, void* Kc, void* Vc, tb_stream_t stream) {
  const NvtxRange range("tb_gather_kv");
  EvictParams p;
  const tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (!idx || !K || !V || !Kc || !Vc) return TB_ERR_INVALID_ARG;
  if (!aligned16(idx) || !aligned16(K) || !aligned16(V) || !aligned16(Kc) || !aligned16(Vc))
    return TB_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return cuda_status(launch_gather(p, idx, K, V, Kc, Vc, nullptr, s));
}

tb_status tb_score_evict(const tb_evict_desc* desc, const void* q_win, const void* K,
                         const void* V, int32_t* idx, void* Kc, void* Vc, float* pooled,
                         void* workspace, size_t workspace_bytes, tb_stream_t stream) {
  const NvtxRange range("tb_score_evict");
  EvictParams p;
  tb_status st = build_evict(desc, &p);
  if (st != TB_OK) return st;
  if (!q_win || !K || !V || !idx || !Kc || !Vc) return TB_ERR_INVALID_ARG;
  if (!aligned16(q_win) || !aligned16(K) || !aligned16(V) || !aligned16(idx) ||
      !aligned16(Kc) || !aligned16(Vc) || (pooled && !aligned16(pooled)))
    return TB_ERR_INVALID_ARG;
  const EvictWorkspace w = carve_evict(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = cuda_status(clear_control_words(workspace, evict_clear_bytes(p, w), s))) != TB_OK) return st;
  float* scores = at<float>(workspace, w.scores);
  if ((st = run_window_scores(p, w, q_win, K, scores, workspace, s)) != TB_OK) return st;
  if ((st = run_select(p, w, scores, idx, pooled, workspace, s)) != TB_OK) return st;
  p.flags &= ~TB_EVICT_GATHER_CONCURRENT;  // this gather reads the select's indices
  return cuda_status(launch_gather(p, idx, K, V, Kc, Vc, at<int32_t>(workspace, w.status), s));
}

tb_status tb_decode_workspace_size(const tb_decode_desc* desc, size_t* bytes) {
  if (!bytes) return TB_ERR_INVALID_ARG;
  DecodeParams p;
  const tb_status st = build_decode(desc, &p);
  if (st != TB_OK) return st;
  *bytes = carve_decode(p).total;
  return TB_OK;
}

tb_status tb_decode_attn(const tb_decode_desc* desc, const void* q, const void* Kc,
                         const void* Vc, const int32_t* lens, void* out, void* workspace,
                         size_t workspace_bytes, tb_stream_t stream) {
  const NvtxRange range("tb_decode_attn");
  DecodeParams p;
  tb_status st = build_decode(desc, &p);
  if (st != TB_OK) return st;
  if (!q || !Kc || !Vc || !lens || !out) return TB_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(Kc) || !aligned16(Vc) || !aligned16(out))
    return TB_ERR_INVALID_ARG;
  const DecodeWorkspace w = carve_decode(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((st = cuda_status(clear_control_words(workspace, w.part_o, s))) != TB_OK) return st;
  return cuda_status(launch_decode(p, q, Kc, Vc, lens, out, at<float>(workspace, w.part_o),
                                   at<float2>(workspace, w.part_ml),
                                   at<int32_t>(workspace, w.counters),
                                   at<int32_t>(workspace, w.status), s));
}

tb_status tb_decode_workspace_prepare(const tb_decode_desc* desc, void* workspace,
                                      size_t workspace_bytes, tb_stream_t stream) {
  const NvtxRange range("tb_decode_workspace_prepare");
  DecodeParams p;
  tb_status st = build_decode(desc, &p);
  if (st != TB_OK) return st;
  const DecodeWorkspace w = carve_decode(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  return cuda_status(
      clear_control_words(workspace, w.part_o, reinterpret_cast<cudaStream_t>(stream)));
}

tb_status tb_decode_attn_prepared(const tb_decode_desc* desc, const void* q, const void* Kc,
                                  const void* Vc, const int32_t* lens, void* out, void* workspace,
                                  size_t workspace_bytes, tb_stream_t stream) {
  const NvtxRange range("tb_decode_attn_prepared");
  DecodeParams p;
  tb_status st = build_decode(desc, &p);
  if (st != TB_OK) return st;
  if (!q || !Kc || !Vc || !lens || !out) return TB_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(Kc) || !aligned16(Vc) || !aligned16(out))
    return TB_ERR_INVALID_ARG;
  const DecodeWorkspace w = carve_decode(p);
  if ((st = check_ws(workspace, workspace_bytes, w.total)) != TB_OK) return st;
  // no clearing kernel: the split counters are zero since the workspace was
  // prepared (each call's last split CTA zeroes its counter again), and the
  // status word keeps what earlier calls raised. Any kernel may precede this
  // one, so its first tiles wait for it, unless the caller asserts that the
  // preceding work writes no cache row below the last appended one (mode 2),
  // or that it writes nothing this call reads and needs no wait at all (3)
  p.early_tma = (desc->flags & TB_DECODE_CONCURRENT)         ? 3
                : (desc->flags & TB_DECODE_EARLY_CACHE_READ) ? 2
                                                             : 0;
  return cuda_status(launch_decode(p, q, Kc, Vc, lens, out, at<float>(workspace, w.part_o),
                                   at<float2>(workspace, w.part_ml),
                                   at<int32_t>(workspace, w.counters),
                                   at<int32_t>(workspace, w.status),
                                   reinterpret_cast<cudaStream_t>(stream)));
}

tb_status tb_read_status(const void* workspace, size_t workspace_bytes, tb_stream_t stream,
                         int32_t* raw) {
  if (!workspace || workspace_bytes < sizeof(int32_t)) return TB_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  tb_status st = cuda_status(cudaStreamSynchronize(s));
  if (st != TB_OK) return st;
  int32_t word = 0;
  st = cuda_status(cudaMemcpy(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost));
  if (st != TB_OK) return st;
  if (raw) *raw = word;
  if (word & kStatusTimeout) return TB_ERR_TIMEOUT;
  if (word & kStatusRange) return TB_ERR_INVALID_ARG;
  return TB_OK;
}

}  // extern "C"
