// Decode-step attention over the compacted GQA cache, split along the keys.
//
// For request b and query head h (KV head g = h / G):
//   out[b][h] = sum_{r < len_b} softmax_r(q[b][h] . Kc[g][r] / sqrt(d)) Vc[g][r]
// (attention definition of "FLOPs-based Modeling" with a single query row;
// len_b = N_kv of Eq. 8). Each CTA takes one (request, KV head, key split),
// keeps the G query heads of the group in shared memory and streams the
// split's K/V tiles once, so every K/V byte is read once for all G heads.
// The split's partial (max, sum, unnormalised output) goes to the workspace
// and a second kernel merges the splits.
#include <cuda_runtime.h>
#include <math.h>

#include "tb_internal.cuh"

namespace tb {
namespace {

constexpr int kDecThreads = 128;
constexpr int kTile = 32;

__device__ __forceinline__ int clamp_len(const DecodeParams& p, const int32_t* lens, int b,
                                         int32_t* status, bool report) {
  int len = lens[b];
  const int64_t cap64 = p.max_len < (int64_t)p.cache_cap[b] ? p.max_len : (int64_t)p.cache_cap[b];
  const int cap = (int)cap64;
  if (len > cap) {
    if (report) atomicOr(status, kStatusRange);
    len = cap;
  }
  return len < 0 ? 0 : len;
}

template <typename T, int D, int GM>
__global__ void __launch_bounds__(kDecThreads) decode_split_simt(
    const __grid_constant__ DecodeParams p, const T* __restrict__ q, const T* __restrict__ Kc,
    const T* __restrict__ Vc, const int32_t* __restrict__ lens, float* __restrict__ part_o,
    float2* __restrict__ part_ml, int32_t* __restrict__ status) {
  constexpr int HS = kDecThreads / D;  // head subsets (1 for d=128, 2 for d=64)
  extern __shared__ float smem[];
  const int G = p.group;
  float* qs = smem;                          // [G][D]
  float* Ks = qs + G * D;                    // [kTile][D + 1]
  float* Vs = Ks + kTile * (D + 1);          // [kTile][D]
  float* ps = Vs + kTile * D;                // [G][kTile]
  float* corr = ps + G * kTile;              // [G]
  float* mrun = corr + G;                    // [G]
  float* lrun = mrun + G;                    // [G]

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int len = clamp_len(p, lens, b, status, split == 0 && g == 0 && tid == 0);
  const int k0 = split * p.split_len;
  const int k1 = min(len, k0 + p.split_len);
  const size_t part_base = ((size_t)b * p.hq + (size_t)g * G) * p.splits + split;

  const int dim = tid % D, hsub = tid / D;
  if (k0 >= k1) {
    for (int hl = hsub; hl < G; hl += HS) {
      part_o[(part_base + (size_t)hl * p.splits) * D + dim] = 0.f;
      if (dim == 0) part_ml[part_base + (size_t)hl * p.splits] = make_float2(-INFINITY, 0.f);
    }
    return;
  }

  const T* qg = q + ((size_t)b * p.hq + (size_t)g * G) * D;
  for (int e = tid; e < G * D; e += kDecThreads) qs[e] = to_f32<T>(qg[e]);
  for (int e = tid; e < G; e += kDecThreads) { mrun[e] = -INFINITY; lrun[e] = 0.f; }
  const T* Kg = Kc + ((size_t)g * p.cache_rows + p.cache_off[b]) * D;
  const T* Vg = Vc + ((size_t)g * p.cache_rows + p.cache_off[b]) * D;

  float acc[GM];
#pragma unroll
  for (int i = 0; i < GM; ++i) acc[i] = 0.f;

  for (int jt = k0; jt < k1; jt += kTile) {
    const int nk = min(kTile, k1 - jt);
    __syncthreads();
    for (int e = tid; e < kTile * D; e += kDecThreads) {
      const int r = e / D, i = e % D;
      const bool ok = r < nk;
      Ks[r * (D + 1) + i] = ok ? to_f32<T>(Kg[(size_t)(jt + r) * D + i]) : 0.f;
      Vs[r * D + i] = ok ? to_f32<T>(Vg[(size_t)(jt + r) * D + i]) : 0.f;
    }
    __syncthreads();
    for (int e = tid; e < G * kTile; e += kDecThreads) {
      const int hl = e / kTile, jj = e % kTile;
      float dot = 0.f;
#pragma unroll 16
      for (int i = 0; i < D; ++i) dot = fmaf(qs[hl * D + i], Ks[jj * (D + 1) + i], dot);
      ps[e] = jj < nk ? dot * p.scale_log2 : -INFINITY;
    }
    __syncthreads();
    for (int hl = warp; hl < G; hl += kDecThreads / 32) {
      const float v = ps[hl * kTile + lane];
      float tmax = v;
      for (int off = 16; off > 0; off >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, off));
      const float m_old = mrun[hl];
      const float m_new = fmaxf(m_old, tmax);
      const float pv = exp2f(v - m_new);
      float sum = pv;
      for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
      ps[hl * kTile + lane] = pv;
      __syncwarp();
      if (lane == 0) {
        const float c = exp2f(m_old - m_new);
        corr[hl] = c;
        lrun[hl] = lrun[hl] * c + sum;
        mrun[hl] = m_new;
      }
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < GM; ++i) {
      const int hl = hsub + HS * i;
      if (hl < G) {
        float a = acc[i] * corr[hl];
        for (int jj = 0; jj < nk; ++jj) a = fmaf(ps[hl * kTile + jj], Vs[jj * D + dim], a);
        acc[i] = a;
      }
    }
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < GM; ++i) {
    const int hl = hsub + HS * i;
    if (hl < G) {
      part_o[(part_base + (size_t)hl * p.splits) * D + dim] = acc[i];
      if (dim == 0) part_ml[part_base + (size_t)hl * p.splits] = make_float2(mrun[hl], lrun[hl]);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(D) decode_combine(const __grid_constant__ DecodeParams p,
                                                    const float* __restrict__ part_o,
                                                    const float2* __restrict__ part_ml,
                                                    void* __restrict__ out) {
  const int h = blockIdx.x, b = blockIdx.y, dim = threadIdx.x;
  const size_t base = ((size_t)b * p.hq + h) * p.splits;
  float m = -INFINITY;
  for (int s = 0; s < p.splits; ++s) m = fmaxf(m, part_ml[base + s].x);
  float l = 0.f, o = 0.f;
  if (m != -INFINITY) {
    for (int s = 0; s < p.splits; ++s) {
      const float2 ml = part_ml[base + s];
      if (ml.y > 0.f) {
        const float w = exp2f(ml.x - m);
        l = fmaf(ml.y, w, l);
        o = fmaf(part_o[(base + s) * D + dim], w, o);
      }
    }
  }
  const float r = l > 0.f ? o / l : 0.f;
  const size_t oi = ((size_t)b * p.hq + h) * D + dim;
  if (p.out_dtype == TB_F32) {
    static_cast<float*>(out)[oi] = r;
  } else {
    static_cast<uint16_t*>(out)[oi] = float_to_bf16_rne(r);
  }
}

template <typename T, int D, int GM>
cudaError_t launch_split(const DecodeParams& p, const void* q, const void* Kc, const void* Vc,
                         const int32_t* lens, void* out, float* part_o, float2* part_ml,
                         int32_t* status, cudaStream_t s) {
  const int G = p.group;
  const size_t smem =
      sizeof(float) * ((size_t)G * D + kTile * (D + 1) + kTile * D + (size_t)G * kTile + 3 * G);
  auto kern = decode_split_simt<T, D, GM>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(p.splits, p.hkv, p.batch);
  kern<<<grid, kDecThreads, smem, s>>>(p, static_cast<const T*>(q), static_cast<const T*>(Kc),
                                       static_cast<const T*>(Vc), lens, part_o, part_ml, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  decode_combine<D><<<dim3(p.hq, p.batch), D, 0, s>>>(p, part_o, part_ml, out);
  count_launches(2);
  return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_d(const DecodeParams& p, const void* q, const void* Kc, const void* Vc,
                     const int32_t* lens, void* out, float* part_o, float2* part_ml,
                     int32_t* status, cudaStream_t s) {
  constexpr int HS = kDecThreads / D;
  const int per_thread = (p.group + HS - 1) / HS;
  if (per_thread <= 4) return launch_split<T, D, 4>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
  if (per_thread <= 8) return launch_split<T, D, 8>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
  if (per_thread <= 16) return launch_split<T, D, 16>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
  return launch_split<T, D, 32>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
}

}  // namespace

cudaError_t launch_decode(const DecodeParams& p, const void* q, const void* Kc, const void* Vc,
                          const int32_t* lens, void* out, float* part_o, float2* part_ml,
                          int32_t* counters, int32_t* status, cudaStream_t s) {
  if (decode_tma_supported(p))
    return launch_decode_tma(p, q, Kc, Vc, lens, part_o, part_ml, counters, out, status, s);
  if (p.dtype == TB_F32) {
    return p.d == 64 ? launch_d<float, 64>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s)
                     : launch_d<float, 128>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
  }
  return p.d == 64 ? launch_d<uint16_t, 64>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s)
                   : launch_d<uint16_t, 128>(p, q, Kc, Vc, lens, out, part_o, part_ml, status, s);
}

}  // namespace tb
