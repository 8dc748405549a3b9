// Decode-step attention over the compacted bf16 cache, TMA-staged.
//
// Same result as the portable kernel in k_decode.cu (one query per head,
// softmax over the request's first len keys, attention definition of
// "FLOPs-based Modeling"), organised for HBM bandwidth: each CTA takes one
// (request, KV head, key split) and streams its K and V rows through a
// 3-stage ring of 64-key tiles that one thread fills with 2-D TMA copies
// (128-byte swizzle, so that reading a key row or a value column from shared
// memory is free of bank conflicts). The G query heads of the group share
// every tile, so each K/V byte is read from HBM once per decode step.
//
// Per 64-key tile (128 threads):
//   scores   thread pair (2i, 2i+1) owns key i, each half of the head dim;
//            q . k for the G heads in fp32, pair-combined with one shuffle;
//   softmax  per-head tile max across the CTA, running max / rescale (log2
//            domain), p = 2^(t - m) written to shared memory;
//   p . V    thread t owns two dims of the output for all heads and half of
//            the tile's keys; the halves are added at the end.
// Partial (max, sum, unnormalised output) per split go to the workspace; the
// CTA that finishes last among a (request, KV head)'s splits (a counter in
// the workspace, zeroed by every call) merges them and writes the output.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>

#include "tb_internal.cuh"
#include "tc_ptx.cuh"

namespace tb {
namespace {

constexpr int kThreads = 128;
constexpr int kTile = 64;
constexpr int kStages = 3;
constexpr int kBox = 64 * 128;  // 64 rows x 128 B

template <int D, int G>
struct DGeo {
  static constexpr int KH = D / 64;
  static constexpr int Gp = (G + 3) & ~3;
  static constexpr int kStageBytes = 2 * KH * kBox;      // K and V halves of one tile
  static constexpr int kRing = kStages * kStageBytes;
  static constexpr int kQOff = kRing;                    // q: G x D floats
  static constexpr int kPOff = kQOff + G * D * 4;        // p: kTile x Gp floats
  static constexpr int kRedOff = kPOff + kTile * Gp * 4; // reductions:
  // per-warp head values (4 x G), then (KPARTS-1) x G x D output parts
  static constexpr int kBarOff = (kRedOff + 4 * G * 4 + G * (256 - D) * 4 + 15) & ~15;
  static constexpr int kSmem = kBarOff + 64 + 1024;      // + alignment slack
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4 v, float (&f)[8]) {
  f[0] = __uint_as_float(v.x << 16);
  f[1] = __uint_as_float(v.x & 0xffff0000u);
  f[2] = __uint_as_float(v.y << 16);
  f[3] = __uint_as_float(v.y & 0xffff0000u);
  f[4] = __uint_as_float(v.z << 16);
  f[5] = __uint_as_float(v.z & 0xffff0000u);
  f[6] = __uint_as_float(v.w << 16);
  f[7] = __uint_as_float(v.w & 0xffff0000u);
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 2)
    decode_tma(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tk,
               const __grid_constant__ CUtensorMap tv, const uint16_t* __restrict__ q,
               const int32_t* __restrict__ lens, float* __restrict__ part_o,
               float2* __restrict__ part_ml, int32_t* __restrict__ counters,
               void* __restrict__ out, int32_t* __restrict__ status) {
  using Gm = DGeo<D, G>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  float* qs = reinterpret_cast<float*>(smem + Gm::kQOff);    // [G][D]
  float* ps = reinterpret_cast<float*>(smem + Gm::kPOff);    // [kTile][Gp]
  float* red = reinterpret_cast<float*>(smem + Gm::kRedOff); // [4 warps][G], then o halves
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Gm::kBarOff);
  int* abort_flag = reinterpret_cast<int*>(smem + Gm::kBarOff + 8 * kStages);
  int* last_flag = abort_flag + 1;
  constexpr int Gp = Gm::Gp;

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int len = lens[b];
  {
    const int64_t cap64 = p.max_len < (int64_t)p.cache_cap[b] ? p.max_len : (int64_t)p.cache_cap[b];
    if (len > (int)cap64) {
      if (split == 0 && g == 0 && tid == 0) atomicOr(status, kStatusRange);
      len = (int)cap64;
    }
    if (len < 0) len = 0;
  }
  const int k0 = split * p.split_len;
  const int k1 = min(len, k0 + p.split_len);
  const size_t part_base = ((size_t)b * p.hq + (size_t)g * G) * p.splits + split;
  const int ntiles = k1 > k0 ? (k1 - k0 + kTile - 1) / kTile : 0;
  const int row0 = (int)((int64_t)g * p.cache_rows + p.cache_off[b]) + k0;

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) tc::mbar_init(&full[s], 1);
    *abort_flag = 0;
    *last_flag = 0;
    tc::fence_barrier_init();
  }
  const uint16_t* qg = q + ((size_t)b * p.hq + (size_t)g * G) * D;
  for (int e = tid; e < G * D; e += kThreads) qs[e] = __uint_as_float((uint32_t)qg[e] << 16);
  __syncthreads();

  auto issue = [&](int t) {
    const int s = t % kStages;
    uint8_t* st = smem + s * Gm::kStageBytes;
    tc::mbar_arrive_expect_tx(&full[s], (uint32_t)Gm::kStageBytes);
    for (int h = 0; h < Gm::KH; ++h) {
      tc::tma_load_2d(st + h * kBox, &tk, h * 64, row0 + t * kTile, &full[s]);
      tc::tma_load_2d(st + (Gm::KH + h) * kBox, &tv, h * 64, row0 + t * kTile, &full[s]);
    }
  };
  int issued = 0;
  if (tid == 0) {
    tc::tma_prefetch_desc(&tk);
    tc::tma_prefetch_desc(&tv);
    for (; issued < kStages && issued < ntiles; ++issued) issue(issued);
  }

  const float c = p.scale_log2;
  // score role: key kk = tid / 2, half hh = tid % 2 of the head dim
  const int kk = tid >> 1, hh = tid & 1;
  // p.V role: dim pair dp (dims 2dp, 2dp+1), key half kh
  constexpr int DP = D / 2;                 // dim pairs
  constexpr int KPARTS = kThreads / DP;     // 2 for d=128, 4 for d=64
  constexpr int KPER = kTile / KPARTS;
  const int dp = tid % DP, kh = tid / DP;
  float m_run[G], l_run[G], o0[G], o1[G];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    m_run[h] = -INFINITY;
    l_run[h] = 0.f;
    o0[h] = 0.f;
    o1[h] = 0.f;
  }
  bool ok = true;

  for (int t = 0; t < ntiles; ++t) {
    const int s = t % kStages;
    const bool got = tc::mbar_wait(&full[s], (uint32_t)((t / kStages) & 1), abort_flag, status);
    if (__syncthreads_or(!got)) {
      ok = false;
      break;
    }
    const uint8_t* kst = smem + s * Gm::kStageBytes;
    const uint8_t* vst = kst + Gm::KH * kBox;
    const int nvalid = min(kTile, k1 - (k0 + t * kTile));

    // ---- scores for key kk, dims of half hh
    float dot[G];
#pragma unroll
    for (int h = 0; h < G; ++h) dot[h] = 0.f;
    constexpr int CH = D / 16;  // 16-byte chunks per half row
#pragma unroll
    for (int c8 = 0; c8 < CH; ++c8) {
      // the two halves start at different 16-byte chunks: no shared bank
      const int cc = D == 128 ? ((c8 + 4 * hh) & 7) : c8;
      const int dim0 = hh * (D / 2) + cc * 8;
      const int box = dim0 >> 6, chunk = (dim0 & 63) >> 3;
      const uint4 raw = *reinterpret_cast<const uint4*>(kst + box * kBox + kk * 128 +
                                                        ((chunk ^ (kk & 7)) << 4));
      float kf[8];
      bf16x8_to_f32(raw, kf);
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float4 qa = *reinterpret_cast<const float4*>(qs + h * D + dim0);
        const float4 qb = *reinterpret_cast<const float4*>(qs + h * D + dim0 + 4);
        float a = dot[h];
        a = fmaf(qa.x, kf[0], a);
        a = fmaf(qa.y, kf[1], a);
        a = fmaf(qa.z, kf[2], a);
        a = fmaf(qa.w, kf[3], a);
        a = fmaf(qb.x, kf[4], a);
        a = fmaf(qb.y, kf[5], a);
        a = fmaf(qb.z, kf[6], a);
        a = fmaf(qb.w, kf[7], a);
        dot[h] = a;
      }
    }
    float tmax[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      dot[h] += __shfl_xor_sync(0xffffffffu, dot[h], 1);
      dot[h] = kk < nvalid ? dot[h] * c : -INFINITY;
      float m = dot[h];
      for (int off = 2; off < 32; off <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
      tmax[h] = m;
    }
    if (lane == 0)
#pragma unroll
      for (int h = 0; h < G; ++h) red[warp * G + h] = tmax[h];
    __syncthreads();
    float corr[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float m_tile = fmaxf(fmaxf(red[h], red[G + h]), fmaxf(red[2 * G + h], red[3 * G + h]));
      const float m_new = fmaxf(m_run[h], m_tile);
      corr[h] = fast_exp2(m_run[h] - m_new);
      m_run[h] = m_new;
      const float pv = fast_exp2(dot[h] - m_new);
      l_run[h] = l_run[h] * corr[h] + (hh == 0 ? pv : 0.f);
      if (hh == 0) ps[kk * Gp + h] = pv;
    }
    __syncthreads();

    // ---- p . V for dims (2dp, 2dp+1), keys kh*KPER .. +KPER
#pragma unroll
    for (int h = 0; h < G; ++h) {
      o0[h] *= corr[h];
      o1[h] *= corr[h];
    }
    const int vbox = (2 * dp) >> 6, vchunk = ((2 * dp) & 63) >> 3, vin = ((2 * dp) & 7) * 2;
#pragma unroll 4
    for (int j = 0; j < KPER; ++j) {
      const int key = kh * KPER + j;
      if (key >= nvalid) break;  // rows past len may hold anything (even NaN)
      const uint32_t v2 = *reinterpret_cast<const uint32_t*>(
          vst + vbox * kBox + key * 128 + ((vchunk ^ (key & 7)) << 4) + vin);
      const float va = __uint_as_float(v2 << 16), vb = __uint_as_float(v2 & 0xffff0000u);
      const float* pk = ps + key * Gp;
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float pw = pk[h];
        o0[h] = fmaf(pw, va, o0[h]);
        o1[h] = fmaf(pw, vb, o1[h]);
      }
    }
    __syncthreads();  // stage s and ps are free again
    if (tid == 0 && issued < ntiles) {
      issue(issued);
      ++issued;
    }
  }

  if (ok && ntiles > 0) {
    // add the key parts of the output, reduce l over the CTA
    float* ored = red + 4 * G;  // [KPARTS-1][G][D]
    if (kh > 0) {
#pragma unroll
      for (int h = 0; h < G; ++h) {
        ored[((kh - 1) * G + h) * D + 2 * dp] = o0[h];
        ored[((kh - 1) * G + h) * D + 2 * dp + 1] = o1[h];
      }
    }
    float lsum[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float v = l_run[h];
      for (int off = 1; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      lsum[h] = v;
    }
    __syncthreads();
    if (lane == 0)
#pragma unroll
      for (int h = 0; h < G; ++h) red[warp * G + h] = lsum[h];
    __syncthreads();
    if (kh == 0) {
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float a = o0[h], bb = o1[h];
        for (int q2 = 1; q2 < KPARTS; ++q2) {
          a += ored[((q2 - 1) * G + h) * D + 2 * dp];
          bb += ored[((q2 - 1) * G + h) * D + 2 * dp + 1];
        }
        float* po = part_o + (part_base + (size_t)h * p.splits) * D;
        po[2 * dp] = a;
        po[2 * dp + 1] = bb;
      }
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      if (tid == h) {
        const float l = red[h] + red[G + h] + red[2 * G + h] + red[3 * G + h];
        part_ml[part_base + (size_t)h * p.splits] = make_float2(m_run[h], l);
      }
    }
  } else if (ok) {  // an empty split: neutral partials
    for (int e = tid; e < G * D; e += kThreads) {
      const int h = e / D, dim = e % D;
      part_o[(part_base + (size_t)h * p.splits) * D + dim] = 0.f;
      if (dim == 0) part_ml[part_base + (size_t)h * p.splits] = make_float2(-INFINITY, 0.f);
    }
  } else if (tid == 0) {
    // drain the copies still in flight before the CTA exits
    int dummy = 0;
    for (int s = 0; s < kStages && s < issued; ++s) {
      const int last = issued - 1 - ((issued - 1 - s) % kStages);
      tc::mbar_wait(&full[s], (uint32_t)((last / kStages) & 1), &dummy, status);
    }
  }
  if (!ok) return;

  // the last split CTA of this (request, KV head) merges every split
  __threadfence();
  __syncthreads();
  if (tid == 0) *last_flag = atomicAdd(&counters[b * p.hkv + g], 1) == p.splits - 1;
  __syncthreads();
  if (!*last_flag) return;
  __threadfence();
  const size_t head0 = ((size_t)b * p.hq + (size_t)g * G) * p.splits;
  for (int e = tid; e < G * D; e += kThreads) {
    const int h = e / D, dim = e % D;
    const size_t hb = head0 + (size_t)h * p.splits;
    float m = -INFINITY;
    for (int sp = 0; sp < p.splits; ++sp) m = fmaxf(m, __ldcg(&part_ml[hb + sp]).x);
    float l = 0.f, o = 0.f;
    if (m != -INFINITY) {
      for (int sp = 0; sp < p.splits; ++sp) {
        const float2 ml = __ldcg(&part_ml[hb + sp]);
        if (ml.y > 0.f) {
          const float wgt = fast_exp2(ml.x - m);
          l = fmaf(ml.y, wgt, l);
          o = fmaf(__ldcg(&part_o[(hb + sp) * D + dim]), wgt, o);
        }
      }
    }
    const float r = l > 0.f ? o / l : 0.f;
    const size_t oi = ((size_t)b * p.hq + (size_t)g * G + h) * D + dim;
    if (p.out_dtype == TB_F32) {
      static_cast<float*>(out)[oi] = r;
    } else {
      static_cast<uint16_t*>(out)[oi] = float_to_bf16_rne(r);
    }
  }
}

template <int D, int G>
cudaError_t launch_g(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                     const void* q, const int32_t* lens, float* part_o, float2* part_ml,
                     int32_t* counters, void* out, int32_t* status, cudaStream_t s) {
  using Gm = DGeo<D, G>;
  auto kern = decode_tma<D, G>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  kern<<<dim3(p.splits, p.hkv, p.batch), kThreads, Gm::kSmem, s>>>(
      p, tk, tv, static_cast<const uint16_t*>(q), lens, part_o, part_ml, counters, out, status);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                     const void* q, const int32_t* lens, float* part_o, float2* part_ml,
                     int32_t* counters, void* out, int32_t* status, cudaStream_t s) {
  switch (p.group) {
#define TB_CASE(GG) \
  case GG:          \
    return launch_g<D, GG>(p, tk, tv, q, lens, part_o, part_ml, counters, out, status, s);
    TB_CASE(1) TB_CASE(2) TB_CASE(3) TB_CASE(4) TB_CASE(5) TB_CASE(6) TB_CASE(7) TB_CASE(8)
    TB_CASE(12) TB_CASE(16)
#undef TB_CASE
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace

bool decode_tma_supported(const DecodeParams& p) {
  const int g = p.group;
  const bool g_ok = (g >= 1 && g <= 8) || g == 12 || g == 16;
  return p.dtype == TB_BF16 && (p.d == 64 || p.d == 128) && g_ok &&
         (uint64_t)p.hkv * (uint64_t)p.cache_rows < (1ull << 31);
}

cudaError_t launch_decode_tma(const DecodeParams& p, const void* q, const void* Kc,
                              const void* Vc, const int32_t* lens, float* part_o,
                              float2* part_ml, int32_t* counters, void* out, int32_t* status,
                              cudaStream_t s) {
  CUtensorMap tk, tv;
  const uint64_t rows = (uint64_t)p.hkv * p.cache_rows;
  if (!make_bf16_map(&tk, Kc, p.d, rows, kTile) || !make_bf16_map(&tv, Vc, p.d, rows, kTile))
    return cudaErrorInvalidValue;
  cudaError_t e =
      p.d == 64 ? launch_d<64>(p, tk, tv, q, lens, part_o, part_ml, counters, out, status, s)
                : launch_d<128>(p, tk, tv, q, lens, part_o, part_ml, counters, out, status, s);
  count_launches(1);
  return e;
}

}  // namespace tb
