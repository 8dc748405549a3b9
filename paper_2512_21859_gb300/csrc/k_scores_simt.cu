// Observation-window scoring, portable SIMT path (fp32 FFMA).
//
// Computes, per request b, KV head g and prefix key j,
//   S[g][j] = sum_{h in g, w < W} exp(s_hwj - m_hw) / l_hw,
//   s_hwj = q_win[h][w] . K[g][j] / sqrt(d),
// where row (h, w) sees keys j <= P + w (causal window) and m_hw, l_hw are
// that row's max and sum of exponentials over its visible keys (the
// attention definition of "FLOPs-based Modeling" restricted to the window
// queries; SnapKV voting per "Experimental Setup").
//
// Three launches: (1) per (request, head, key chunk) partial row statistics,
// (2) a per-row merge into c_hw = log2-sum-exp, (3) the normalised window
// sum per key. Work is in log2 units: t = s * log2(e), p = 2^(t - c).
// fp32 inputs must come here (no TF32 tensor path); bf16 inputs may.
#include <cuda_runtime.h>
#include <math.h>

#include <type_traits>

#include "tb_internal.cuh"

namespace tb {
namespace {

constexpr int kRowsPerBlock = 32;  // query rows staged per pass
constexpr int kKeysPerTile = 32;   // keys staged per tile (one per lane)
constexpr int kWarps = 8;

__device__ __forceinline__ int find_request(const EvictParams& p, int item) {
  int b = 0;
  while (b + 1 < p.batch && p.req[b + 1].item0 <= item) ++b;
  return b;
}

template <typename T, int D>
__device__ __forceinline__ void stage_rows(float (*dst)[D + 1], const T* src, int rows_avail,
                                           int nrows) {
  for (int e = threadIdx.x; e < nrows * D; e += blockDim.x) {
    int r = e / D, i = e % D;
    dst[r][i] = r < rows_avail ? to_f32<T>(src[(size_t)r * D + i]) : 0.f;
  }
}

// (1) partial (max, sum) per window row over one key chunk.
template <typename T, int D>
__global__ void __launch_bounds__(256) ws_stats_simt(const __grid_constant__ EvictParams p,
                                                     const T* __restrict__ q_win,
                                                     const T* __restrict__ K,
                                                     float2* __restrict__ partial) {
  __shared__ float Qs[kRowsPerBlock][D + 1];
  __shared__ float Ks[kKeysPerTile][D + 1];
  const int item = blockIdx.x;
  const int b = find_request(p, item);
  const EvictReq& rq = p.req[b];
  const int nch = (rq.n + p.chunk - 1) / p.chunk;
  const int local = item - rq.item0;
  const int g = local / nch, c = local % nch;
  const int j0 = c * p.chunk, j1 = min(rq.n, j0 + p.chunk);
  const int M = p.m_rows, W = p.window, P = rq.p;
  const T* Kg = K + ((size_t)g * p.kv_rows + rq.kv_off) * D;
  const T* Qg = q_win + ((size_t)b * p.hq + (size_t)g * p.group) * W * D;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  constexpr int RPW = kRowsPerBlock / kWarps;

  for (int rb = 0; rb < M; rb += kRowsPerBlock) {
    __syncthreads();
    stage_rows<T, D>(Qs, Qg + (size_t)rb * D, M - rb, kRowsPerBlock);
    float m[RPW], l[RPW];
#pragma unroll
    for (int i = 0; i < RPW; ++i) { m[i] = -INFINITY; l[i] = 0.f; }
    for (int jt = j0; jt < j1; jt += kKeysPerTile) {
      __syncthreads();
      stage_rows<T, D>(Ks, Kg + (size_t)jt * D, j1 - jt, kKeysPerTile);
      __syncthreads();
      const int j = jt + lane;
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        const int rl = warp * RPW + i, r = rb + rl;
        float dot = 0.f;
#pragma unroll 16
        for (int e = 0; e < D; ++e) dot = fmaf(Qs[rl][e], Ks[lane][e], dot);
        const bool vis = (j < j1) && (r < M) && (j <= P + (r % W));
        if (vis) {
          const float t = dot * p.scale_log2;
          if (t > m[i]) {
            l[i] = l[i] * exp2f(m[i] - t) + 1.f;
            m[i] = t;
          } else {
            l[i] += exp2f(t - m[i]);
          }
        }
      }
    }
    // merge the 32 lanes of each row
#pragma unroll
    for (int i = 0; i < RPW; ++i) {
      float mm = m[i], ll = l[i];
      for (int off = 16; off > 0; off >>= 1) {
        const float mo = __shfl_xor_sync(0xffffffffu, mm, off);
        const float lo = __shfl_xor_sync(0xffffffffu, ll, off);
        const float mn = fmaxf(mm, mo);
        if (mn == -INFINITY) {
          ll = 0.f;
        } else {
          ll = ll * exp2f(mm - mn) + lo * exp2f(mo - mn);
        }
        mm = mn;
      }
      const int r = rb + warp * RPW + i;
      if (lane == 0 && r < M) partial[(size_t)item * M + r] = make_float2(mm, ll);
    }
  }
}

// (2) merge chunk partials: c = m + log2(l), fp32 with a compensated sum.
__global__ void __launch_bounds__(256) ws_combine(const __grid_constant__ EvictParams p,
                                                  const float2* __restrict__ partial,
                                                  float* __restrict__ rowc) {
  const int seg = blockIdx.x;  // b * hkv + g
  const int b = seg / p.hkv, g = seg % p.hkv;
  const EvictReq& rq = p.req[b];
  const int nch = (rq.n + p.chunk - 1) / p.chunk;
  const int M = p.m_rows;
  const size_t item0 = (size_t)rq.item0 + (size_t)g * nch;
  for (int r = threadIdx.x; r < M; r += blockDim.x) {
    float m = -INFINITY;
    for (int c = 0; c < nch; ++c) m = fmaxf(m, partial[(item0 + c) * M + r].x);
    float l = 0.f, comp = 0.f;  // compensated (Kahan) sum
    for (int c = 0; c < nch; ++c) {
      const float2 v = partial[(item0 + c) * M + r];
      if (v.y > 0.f) {
        const float term = v.y * exp2f(v.x - m) - comp;
        const float t = l + term;
        comp = (t - l) - term;
        l = t;
      }
    }
    rowc[(size_t)seg * M + r] = m + log2f(l);
  }
}

// (3) normalised window sum per prefix key.
template <typename T, int D>
__global__ void __launch_bounds__(256) ws_scores_simt(const __grid_constant__ EvictParams p,
                                                      const T* __restrict__ q_win,
                                                      const T* __restrict__ K,
                                                      const float* __restrict__ rowc,
                                                      float* __restrict__ scores) {
  __shared__ float Qs[kRowsPerBlock][D + 1];
  __shared__ float Ks[kKeysPerTile][D + 1];
  __shared__ float Cs[kRowsPerBlock];
  __shared__ float part[kWarps][kSimtChunk];
  const int item = blockIdx.x;
  const int b = find_request(p, item);
  const EvictReq& rq = p.req[b];
  const int nch = (rq.n + p.chunk - 1) / p.chunk;
  const int local = item - rq.item0;
  const int g = local / nch, c = local % nch;
  const int P = rq.p;
  const int j0 = c * p.chunk, j1 = min(P, j0 + p.chunk);
  if (j0 >= j1) return;  // chunk holds window keys only
  const int M = p.m_rows, W = p.window;
  const T* Kg = K + ((size_t)g * p.kv_rows + rq.kv_off) * D;
  const T* Qg = q_win + ((size_t)b * p.hq + (size_t)g * p.group) * W * D;
  const float* Cg = rowc + ((size_t)b * p.hkv + g) * M;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  constexpr int RPW = kRowsPerBlock / kWarps;

  for (int e = threadIdx.x; e < kWarps * kSimtChunk; e += blockDim.x) (&part[0][0])[e] = 0.f;
  for (int rb = 0; rb < M; rb += kRowsPerBlock) {
    __syncthreads();
    stage_rows<T, D>(Qs, Qg + (size_t)rb * D, M - rb, kRowsPerBlock);
    for (int e = threadIdx.x; e < kRowsPerBlock; e += blockDim.x)
      Cs[e] = rb + e < M ? Cg[rb + e] * p.rowc_scale : 0.f;
    for (int jt = j0; jt < j1; jt += kKeysPerTile) {
      __syncthreads();
      stage_rows<T, D>(Ks, Kg + (size_t)jt * D, j1 - jt, kKeysPerTile);
      __syncthreads();
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        const int rl = warp * RPW + i;
        float dot = 0.f;
#pragma unroll 16
        for (int e = 0; e < D; ++e) dot = fmaf(Qs[rl][e], Ks[lane][e], dot);
        if (rb + rl < M) acc += exp2f(dot * p.scale_log2 - Cs[rl]);
      }
      if (jt + lane < j1) part[warp][jt - j0 + lane] += acc;
    }
  }
  __syncthreads();
  float* out = scores + (size_t)g * p.score_rows + rq.score_off;
  for (int j = j0 + threadIdx.x; j < j1; j += blockDim.x) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += part[w][j - j0];
    out[j] = s;
  }
}

template <typename T, int D>
cudaError_t launch_typed(const EvictParams& p, const void* q_win, const void* K, float* scores,
                         float2* partial, float* rowc, cudaStream_t s) {
  ws_stats_simt<T, D><<<p.items, 256, 0, s>>>(p, static_cast<const T*>(q_win),
                                              static_cast<const T*>(K), partial);
  ws_combine<<<p.batch * p.hkv, 256, 0, s>>>(p, partial, rowc);
  ws_scores_simt<T, D><<<p.items, 256, 0, s>>>(p, static_cast<const T*>(q_win),
                                               static_cast<const T*>(K), rowc, scores);
  count_launches(3);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_window_combine(const EvictParams& p, const float2* partial, float* rowc,
                                  cudaStream_t s) {
  ws_combine<<<p.batch * p.hkv, 256, 0, s>>>(p, partial, rowc);
  count_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_window_votes_simt(const EvictParams& p, const void* q_win, const void* K,
                                     float* scores, const float* rowc, cudaStream_t s) {
  auto go = [&](auto kern, auto qt) {
    using T = std::remove_const_t<std::remove_pointer_t<decltype(qt)>>;
    kern<<<p.items, 256, 0, s>>>(p, static_cast<const T*>(q_win), static_cast<const T*>(K), rowc,
                                 scores);
    count_launches(1);
    return cudaGetLastError();
  };
  if (p.dtype == TB_F32)
    return p.d == 64 ? go(ws_scores_simt<float, 64>, (const float*)nullptr)
                     : go(ws_scores_simt<float, 128>, (const float*)nullptr);
  return p.d == 64 ? go(ws_scores_simt<uint16_t, 64>, (const uint16_t*)nullptr)
                   : go(ws_scores_simt<uint16_t, 128>, (const uint16_t*)nullptr);
}

cudaError_t launch_window_scores_simt(const EvictParams& p, const void* q_win, const void* K,
                                      float* scores, float2* partial, float* rowc,
                                      cudaStream_t s) {
  if (p.dtype == TB_F32) {
    return p.d == 64 ? launch_typed<float, 64>(p, q_win, K, scores, partial, rowc, s)
                     : launch_typed<float, 128>(p, q_win, K, scores, partial, rowc, s);
  }
  return p.d == 64 ? launch_typed<uint16_t, 64>(p, q_win, K, scores, partial, rowc, s)
                   : launch_typed<uint16_t, 128>(p, q_win, K, scores, partial, rowc, s);
}

}  // namespace tb
