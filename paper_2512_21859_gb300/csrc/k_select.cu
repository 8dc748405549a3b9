// Max-pool and per-head top-k selection with ordered compaction.
//
// Pool[j] = max of S over [j - pool_k/2, j + pool_k/2] clipped to the prefix
// (stride 1, out-of-range neighbours ignored). Then, per (request, KV head),
// the k largest pooled scores are kept, ties to the lower index, and written
// in ascending index order followed by the window positions P..N-1.
//
// Selection is a most-significant-digit radix select on the float bit
// pattern (scores are >= 0, so unsigned order equals numeric order): four
// 8-bit digit histograms find the k-th largest value tau and how many of the
// tau-valued entries to keep; one ordered pass then keeps every entry above
// tau and the first `need` entries equal to tau, which yields sorted indices
// without a sort.
#include <cuda_runtime.h>

#include "tb_internal.cuh"

namespace tb {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;

__global__ void __launch_bounds__(256) pool_kernel(const __grid_constant__ EvictParams p,
                                                   const float* __restrict__ scores,
                                                   float* __restrict__ pooled) {
  const int b = blockIdx.y, g = blockIdx.z;
  const EvictReq& rq = p.req[b];
  const int P = rq.p, half = p.pool_k / 2;
  const size_t base = (size_t)g * p.score_rows + rq.score_off;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < P; j += gridDim.x * blockDim.x) {
    const int lo = max(0, j - half), hi = min(P - 1, j + half);
    float m = scores[base + lo];
    for (int t = lo + 1; t <= hi; ++t) m = fmaxf(m, scores[base + t]);
    pooled[base + j] = m;
  }
}

// Block-wide exclusive scan of a 0/1 flag; returns the prefix, sets *total.
__device__ __forceinline__ int block_scan_flag(bool flag, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned ball = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(ball & ((1u << lane) - 1u));
  if (lane == 0) warp_tot[warp] = __popc(ball);
  __syncthreads();
  if (warp == 0) {
    const int v = lane < kSelWarps ? warp_tot[lane] : 0;
    int inc = v;
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += o;
    }
    if (lane < kSelWarps) warp_tot[lane] = inc - v;  // exclusive
    if (lane == 31) warp_tot[32] = inc;
  }
  __syncthreads();
  const int res = warp_tot[warp] + in_warp;
  *total = warp_tot[32];
  __syncthreads();
  return res;
}

__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ EvictParams p,
                                                             const float* __restrict__ pooled,
                                                             int32_t* __restrict__ idx) {
  __shared__ unsigned hist[256];
  __shared__ int warp_tot[33];
  __shared__ unsigned sh_prefix;
  __shared__ int sh_need;
  const int b = blockIdx.x / p.hkv, g = blockIdx.x % p.hkv;
  const EvictReq& rq = p.req[b];
  const int P = rq.p, k = rq.k;
  const unsigned* key = reinterpret_cast<const unsigned*>(pooled + (size_t)g * p.score_rows +
                                                          rq.score_off);
  int32_t* out = idx + (size_t)g * p.idx_rows + rq.idx_off;
  const int tid = threadIdx.x;

  for (int t = tid; t < p.window; t += blockDim.x) out[k + t] = P + t;
  if (k == 0) return;
  if (k >= P) {
    for (int j = tid; j < P; j += blockDim.x) out[j] = j;
    return;
  }

  // radix select of the k-th largest key, most significant digit first
  unsigned prefix = 0, mask = 0;
  int need = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int t = tid; t < 256; t += blockDim.x) hist[t] = 0;
    __syncthreads();
    for (int j = tid; j < P; j += blockDim.x) {
      const unsigned u = key[j];
      if ((u & mask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      // warp 0: find the digit where the count from the top reaches `need`
      unsigned above = 0;  // entries with a larger digit than this lane's block
      // lanes own 8 digits each, highest digits on lane 0
      unsigned cnt[8];
      unsigned mine = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        cnt[i] = hist[255 - (tid * 8 + i)];
        mine += cnt[i];
      }
      unsigned inc = mine;
      for (int off = 1; off < 32; off <<= 1) {
        const unsigned o = __shfl_up_sync(0xffffffffu, inc, off);
        if (tid >= off) inc += o;
      }
      above = inc - mine;
      if (above < (unsigned)need && inc >= (unsigned)need) {
        unsigned run = above;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (run + cnt[i] >= (unsigned)need) {
            const unsigned digit = 255u - (unsigned)(tid * 8 + i);
            sh_prefix = prefix | (digit << shift);
            sh_need = need - (int)run;
            break;
          }
          run += cnt[i];
        }
      }
    }
    __syncthreads();
    prefix = sh_prefix;
    need = sh_need;
    mask |= 255u << shift;
    __syncthreads();
  }
  const unsigned tau = prefix;  // `need` entries equal to tau are kept

  int base_sel = 0, base_tie = 0;
  for (int s = 0; s < P; s += blockDim.x) {
    const int j = s + tid;
    const unsigned u = j < P ? key[j] : 0u;
    const bool gt = j < P && u > tau;
    const bool eq = j < P && u == tau;
    int tot_eq;
    const int tie_rank = base_tie + block_scan_flag(eq, warp_tot, &tot_eq);
    const bool sel = gt || (eq && tie_rank < need);
    int tot_sel;
    const int pos = base_sel + block_scan_flag(sel, warp_tot, &tot_sel);
    if (sel && pos < k) out[pos] = j;
    base_sel += tot_sel;
    base_tie += tot_eq;
  }
}

}  // namespace

cudaError_t launch_pool(const EvictParams& p, const float* scores, float* pooled, cudaStream_t s) {
  const int bx = (p.max_p + 255) / 256;
  if (bx == 0) return cudaSuccess;
  dim3 grid(bx < 1024 ? bx : 1024, p.batch, p.hkv);
  pool_kernel<<<grid, 256, 0, s>>>(p, scores, pooled);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_select(const EvictParams& p, const float* pooled, int32_t* idx,
                          cudaStream_t s) {
  select_kernel<<<p.batch * p.hkv, kSelThreads, 0, s>>>(p, pooled, idx);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace tb
