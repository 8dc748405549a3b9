// Decode-step attention over the compacted bf16 cache, TMA-staged, on
// mma.sync tensor-core fragments.
//
// Same result as the portable kernel in k_decode.cu (one query per head,
// softmax over the request's first len keys, attention definition of
// "FLOPs-based Modeling"), organised for HBM bandwidth: each CTA takes one
// (request, KV head, key split) and streams its K and V rows through a
// 3-stage ring of 128-key tiles that one thread fills with 2-D TMA copies
// (128-byte swizzle, so ldmatrix reads are free of bank conflicts). The G
// query heads of the group share every tile, so each K/V byte is read from
// HBM once per decode step.
//
// Warp w owns keys [16w, 16w + 16) of every tile and keeps its own running
// max / sum / output for the G heads (rows of a 16-row MMA tile; rows past G
// are zero queries whose results are dropped):
//   S = Q K^T      mma.m16n8k16 bf16 -> fp32, K fragments by ldmatrix;
//   softmax        per row over the warp's keys, log2 domain, fp32;
//   O += P V       P in fp32 is split into a bf16 part and a bf16 residual,
//                  both multiplied by V (ldmatrix.trans) and accumulated in
//                  fp32, so P enters with ~16 significant bits.
// At the end the eight warps merge in shared memory into the split's partial
// (max, sum, unnormalised output); the CTA that finishes last among a
// (request, KV head)'s splits (a counter in the workspace: zero before the
// call, and set back to zero by that CTA) merges the splits and writes the
// output.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>

#include "tb_internal.cuh"
#include "tc_ptx.cuh"

namespace tb {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kTile = kWarps * 16;  // keys per tile: 16 per warp
constexpr int kStages = 3;          // one CTA per SM, 3 x 64 KB in flight
constexpr int kBox = kTile * 128;   // one TMA box: kTile rows x 128 B
#ifndef TB_MERGE_PARTS
#define TB_MERGE_PARTS 4
#endif
constexpr int kMergeParts = TB_MERGE_PARTS;  // CTAs of the merge kernel per (KV head, request)

template <int D>
struct DGeo {
  static constexpr int KH = D / 64;
  static constexpr int kStageBytes = 2 * KH * kBox;  // K and V halves of one tile
  static constexpr int kRing = kStages * kStageBytes;
  // after the key loop the ring holds the cross-warp merge: O, m, l per warp
  // (rows padded by 8 floats so the fragment stores hit distinct banks)
  static constexpr int kDS = D + 8;
  static constexpr int kMergeO = kWarps * 16 * kDS * 4;
  // O, (m, l) per warp, then the per-head warp weights [16][kWarps]
  static_assert(kMergeO + kWarps * 16 * 8 + 16 * kWarps * 4 <= kRing,
                "merge area must fit in the ring");
  static constexpr int kMaxSplits = kRing / (16 * 4);  // weights table [G <= 16][splits]
  static constexpr int kBarOff = kRing;
  static constexpr int kSmem = kBarOff + 64 + 1024;  // + alignment slack
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// c (16x8 fp32) += a (16x16 bf16, row) * b (16x8 bf16, col)
__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// two fp32 -> bf16x2 (lo in the low half), round to nearest even
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// byte offset of 16-byte chunk `chunk` (of the D/8 in a row) of tile row `row`
// inside a stage half (K or V) laid out as KH boxes of 64 rows x 128 B, 128B-swizzled
__device__ __forceinline__ uint32_t sw_off(int row, int chunk) {
  return (uint32_t)((chunk >> 3) * kBox + row * 128 + (((chunk & 7) ^ (row & 7)) << 4));
}

// Merges the key splits of (request b, KV head g) into the output: per head
// the weight 2^(m_s - M) / L of every split s, then each output element as
// one pass over the splits' unnormalised partial outputs: the dims of part
// `dpart` of DS equal parts. wts: shared memory for [G][splits] floats.
template <int D, int G, int DS>
__device__ __forceinline__ void merge_splits(const DecodeParams& p, int b, int g, int dpart,
                                             const float* __restrict__ part_o,
                                             const float2* __restrict__ part_ml,
                                             void* __restrict__ out, int32_t* __restrict__ status,
                                             float* wts, int len) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const size_t head0 = ((size_t)b * p.hq + (size_t)g * G) * p.splits;
  // outputs in float4 groups of dims; the splits are divided among the
  // threads that share an output (NS of them), their sums combined by shuffles
  constexpr int D4 = D / 4 / DS;  // float4 groups of this part
  const int d4_0 = dpart * D4;
  // (G * D4 * NS is a multiple of 32 for every supported G and D, so each
  // warp's lanes run the same iterations and the shuffles see full warps)
  constexpr int kPer = kThreads / (G * D4);
  constexpr int NS = kPer >= 8 ? 8 : kPer >= 4 ? 4 : kPer >= 2 ? 2 : 1;
  static_assert((G * D4 * NS) % 32 == 0, "output groups must fill whole warps");
  // Each thread's partial outputs are loaded kChunk splits at a time, all in
  // flight together; the first chunk of its first output group is requested
  // before the split weights are computed, so that those loads and the
  // (max, sum) loads travel at once.
  // (one chunk covers the ~38 splits per thread of one request with four KV
  // heads; with NS > 1 each thread has about half as many)
  constexpr int kChunk = NS >= 2 ? 16 : 40;
  float4 ov[kChunk];
  {
    const int e0 = tid, e = e0 / NS, part = e0 % NS;
    const int h = e / D4, d4 = d4_0 + e % D4;
#pragma unroll
    for (int c = 0; c < kChunk; ++c) {
      const int sp = part + c * NS;
      ov[c] = (e0 < G * D4 * NS && sp < p.splits)
                  ? __ldcg(reinterpret_cast<const float4*>(
                               part_o + (head0 + (size_t)h * p.splits + sp) * D) +
                           d4)
                  : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  // per head: weight of split s = 2^(m_s - M) / L, lanes over splits; the
  // (m, l) pairs of the first 64 splits are loaded once and kept
  for (int h = warp; h < G; h += kThreads / 32) {
    const size_t hb = head0 + (size_t)h * p.splits;
    float2 ml[2];
    float M = -INFINITY;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int sp = lane + 32 * i;
      ml[i] = sp < p.splits ? __ldcg(&part_ml[hb + sp]) : make_float2(-INFINITY, 0.f);
      M = fmaxf(M, ml[i].x);
    }
    for (int sp = lane + 64; sp < p.splits; sp += 32) M = fmaxf(M, __ldcg(&part_ml[hb + sp]).x);
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float L = 0.f;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int sp = lane + 32 * i;
      const float wgt = (M != -INFINITY && ml[i].y > 0.f) ? fast_exp2(ml[i].x - M) : 0.f;
      if (sp < p.splits) wts[h * p.splits + sp] = wgt;
      L = fmaf(ml[i].y, wgt, L);
    }
    for (int sp = lane + 64; sp < p.splits; sp += 32) {
      const float2 m2 = __ldcg(&part_ml[hb + sp]);
      const float wgt = (M != -INFINITY && m2.y > 0.f) ? fast_exp2(m2.x - M) : 0.f;
      wts[h * p.splits + sp] = wgt;
      L = fmaf(m2.y, wgt, L);
    }
    for (int off = 16; off > 0; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
    debug_flag(lane == 0 && len > 0 && !(L > 0.f && isfinite(L)), status);
    const float inv = L > 0.f ? 1.f / L : 0.f;
    __syncwarp();
    for (int sp = lane; sp < p.splits; sp += 32) wts[h * p.splits + sp] *= inv;
  }
  __syncthreads();
  for (int e0 = tid; e0 < G * D4 * NS; e0 += kThreads) {
    const int e = e0 / NS, part = e0 % NS;
    const int h = e / D4, d4 = d4_0 + e % D4;
    const size_t hb = head0 + (size_t)h * p.splits;
    const float* wh = wts + h * p.splits;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    // splits part, part + NS, ... in order, kChunk at a time (the first
    // chunk of the first group is in ov already)
    for (int sp0 = part; sp0 < p.splits; sp0 += kChunk * NS) {
      if (e0 != tid || sp0 != part) {
#pragma unroll
        for (int c = 0; c < kChunk; ++c) {
          const int sp = sp0 + c * NS;
          ov[c] = sp < p.splits ? __ldcg(reinterpret_cast<const float4*>(part_o + (hb + sp) * D) + d4)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
#pragma unroll
      for (int c = 0; c < kChunk; ++c) {
        const int sp = sp0 + c * NS;
        if (sp < p.splits) {
          const float wgt = wh[sp];
          acc.x = fmaf(ov[c].x, wgt, acc.x);
          acc.y = fmaf(ov[c].y, wgt, acc.y);
          acc.z = fmaf(ov[c].z, wgt, acc.z);
          acc.w = fmaf(ov[c].w, wgt, acc.w);
        }
      }
    }
#pragma unroll
    for (int off = 1; off < NS; off <<= 1) {
      acc.x += __shfl_xor_sync(0xffffffffu, acc.x, off);
      acc.y += __shfl_xor_sync(0xffffffffu, acc.y, off);
      acc.z += __shfl_xor_sync(0xffffffffu, acc.z, off);
      acc.w += __shfl_xor_sync(0xffffffffu, acc.w, off);
    }
    if (part != 0) continue;
    const size_t oi = ((size_t)b * p.hq + (size_t)g * G + h) * D + 4 * d4;
    if (p.out_dtype == TB_F32) {
      *reinterpret_cast<float4*>(static_cast<float*>(out) + oi) = acc;
    } else {
      uint16_t* ob = static_cast<uint16_t*>(out) + oi;
      ob[0] = float_to_bf16_rne(acc.x);
      ob[1] = float_to_bf16_rne(acc.y);
      ob[2] = float_to_bf16_rne(acc.z);
      ob[3] = float_to_bf16_rne(acc.w);
    }
  }
}

template <int D, int G>
__device__ __forceinline__ void decode_tma_body(
    const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
    const uint16_t* __restrict__ kc, const uint16_t* __restrict__ vc,
    const uint16_t* __restrict__ q, const int32_t* __restrict__ lens, float* __restrict__ part_o,
    float2* __restrict__ part_ml, int32_t* __restrict__ counters, void* __restrict__ out,
    int32_t* __restrict__ status) {
  using Gm = DGeo<D>;
  constexpr int KS = D / 16;  // k-steps of Q K^T
  constexpr int NT = D / 8;   // n-tiles of P V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Gm::kBarOff);
  int* abort_flag = reinterpret_cast<int*>(smem + Gm::kBarOff + 8 * kStages);
  int* last_flag = abort_flag + 1;

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int r0 = lane >> 2, qd = lane & 3;  // fragment row (and row + 8), column pair
  // The first tiles are requested before the length is read (its load
  // would delay them by a memory round trip): they cover the split's rows up
  // to the request's cap, which lie inside its slice of the cache; tiles
  // past the length are waited for and dropped after the key loop.
  const int k0 = split * p.split_len;
  const int64_t cap64 = p.max_len < (int64_t)p.cache_cap[b] ? p.max_len : (int64_t)p.cache_cap[b];
  const int k1c = (int)min((int64_t)k0 + p.split_len, cap64);
  const int ntiles_c = k1c > k0 ? (k1c - k0 + kTile - 1) / kTile : 0;
  const int row0 = (int)((int64_t)g * p.cache_rows + p.cache_off[b]) + k0;

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) tc::mbar_init(&full[s], 1);
    *abort_flag = 0;
    *last_flag = 0;
    tc::fence_barrier_init();
  }
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
  // With p.early_tma the first tiles are requested before the dependency
  // wait. Mode 1: the kernel launched just before this one on the stream is
  // the library's own clearing kernel (it writes only the workspace's control
  // words), which lets this one start only after its own wait has returned,
  // i.e. once every earlier kernel has completed and its writes are visible;
  // the cache rows cannot be written by the clearing kernel. Mode 2: the
  // caller asserts the same of the work before this kernel for every row
  // below lens[b] - 1; that last row (appended by the decode loop, possibly
  // by the preceding kernel) is read again after the wait, below. Mode 3:
  // the caller asserts that the preceding kernel writes nothing this one
  // reads and that everything it reads was complete before that kernel was
  // launched, so there is no wait before the work and this kernel runs
  // beside it (one thread waits for it at the very end, below).
  // Without either (a prepared workspace, no assertion) any kernel may
  // precede this one, so the requests wait for it.
  int issued = 0;
  if (tid == 0) {
    tc::tma_prefetch_desc(&tk);
    tc::tma_prefetch_desc(&tv);
    if (p.early_tma)
      for (; issued < kStages && issued < ntiles_c; ++issued) issue(issued);
  }
  if (p.early_tma != 3) pdl_wait();
  pdl_trigger();
  if (tid == 0)
    for (; issued < kStages && issued < ntiles_c; ++issued) issue(issued);
  int len = lens[b];
  if (len > (int)cap64) {
    if (split == 0 && g == 0 && tid == 0) atomicOr(status, kStatusRange);
    len = (int)cap64;
  }
  if (len < 0) len = 0;
  const int k1 = min(len, k0 + p.split_len);
  const int ntiles = k1 > k0 ? (k1 - k0 + kTile - 1) / kTile : 0;  // <= ntiles_c
  const size_t part_base = ((size_t)b * p.hq + (size_t)g * G) * p.splits + split;
  // mode 2: the tile (one of those requested before the wait) holding the
  // appended row len - 1, whose copy may predate the row; -1 if none
  const int fresh_key = len - 1 - k0;
  const int fresh_tile = (p.early_tma == 2 && fresh_key >= 0 && fresh_key < k1 - k0 &&
                          fresh_key / kTile < kStages)
                             ? fresh_key / kTile
                             : -1;

  // Q fragments (rows >= G are zero queries)
  uint32_t aq[KS][4];
  {
    const uint32_t* qg = reinterpret_cast<const uint32_t*>(q + ((size_t)b * p.hq + (size_t)g * G) * D);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
      const int w0 = (kk * 16 + 2 * qd) >> 1;  // bf16 pair index in a row
      aq[kk][0] = r0 < G ? qg[r0 * (D / 2) + w0] : 0u;
      aq[kk][1] = r0 + 8 < G ? qg[(r0 + 8) * (D / 2) + w0] : 0u;
      aq[kk][2] = r0 < G ? qg[r0 * (D / 2) + w0 + 4] : 0u;
      aq[kk][3] = r0 + 8 < G ? qg[(r0 + 8) * (D / 2) + w0 + 4] : 0u;
    }
  }

  const float c = p.scale_log2;
  float o[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  const int kb = warp * 16;  // this warp's first key in a tile
  bool ok = true;

  for (int t = 0; t < ntiles; ++t) {
    const int s = t % kStages;
    const bool got = tc::mbar_wait(&full[s], (uint32_t)((t / kStages) & 1), abort_flag, status);
    if (__syncthreads_or(!got)) {
      ok = false;
      break;
    }
    const uint32_t kst = tc::smem_addr(smem + s * Gm::kStageBytes);
    const uint32_t vst = kst + (uint32_t)(Gm::KH * kBox);
    const int nvalid = min(kTile, k1 - (k0 + t * kTile));
    if (t == fresh_tile) {
      // the appended row, read again now that the kernel before this one has
      // completed: the warp that owns it copies its K and V chunks over the
      // tile's (swizzled) copy before reading them
      const int row = fresh_key - t * kTile;
      if ((row >> 4) == warp && lane < 2 * (D / 8)) {
        const int half = lane / (D / 8), chunk = lane % (D / 8);
        const size_t gi = ((size_t)g * p.cache_rows + p.cache_off[b] + (size_t)(k0 + fresh_key)) * D;
        const uint4 v = __ldcg(reinterpret_cast<const uint4*>((half ? vc : kc) + gi) + chunk);
        *reinterpret_cast<uint4*>(smem + s * Gm::kStageBytes + half * (Gm::KH * kBox) +
                                  sw_off(row, chunk)) = v;
      }
      __syncwarp();
    }
    if (kb < nvalid) {
      // rows past len may hold anything (even NaN): clear this warp's V rows there
      if (kb + 16 > nvalid) {
        uint8_t* vrow = smem + s * Gm::kStageBytes + Gm::KH * kBox;
        for (int e = lane; e < (kb + 16 - nvalid) * (D / 8); e += 32) {
          const int row = nvalid + e / (D / 8), chunk = e % (D / 8);
          *reinterpret_cast<uint4*>(vrow + sw_off(row, chunk)) = make_uint4(0, 0, 0, 0);
        }
        __syncwarp();
      }
      // ---- S = Q K^T over this warp's 16 keys
      float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
      {
        // even and odd k-steps accumulate separately: two short dependency
        // chains per n-tile instead of one long one
        float so[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        const int krow = kb + (lane & 7) + ((lane >> 4) << 3);
        const int ksel = (lane >> 3) & 1;
#pragma unroll
        for (int kk = 0; kk < KS; kk += 2) {
          uint32_t bk[4], bk2[4];
          ldsm_x4(kst + sw_off(krow, 2 * kk + ksel), bk);
          ldsm_x4(kst + sw_off(krow, 2 * kk + 2 + ksel), bk2);
          mma_16816(sc[0], aq[kk], bk[0], bk[1]);
          mma_16816(sc[1], aq[kk], bk[2], bk[3]);
          mma_16816(so[0], aq[kk + 1], bk2[0], bk2[1]);
          mma_16816(so[1], aq[kk + 1], bk2[2], bk2[3]);
        }
#pragma unroll
        for (int n = 0; n < 2; ++n)
#pragma unroll
          for (int e = 0; e < 4; ++e) sc[n][e] += so[n][e];
      }
      // ---- online softmax per row (r0: elements 0,1; r0 + 8: elements 2,3)
      float corr[2];
#pragma unroll
      for (int hr = 0; hr < 2; ++hr) {
        float mx = -INFINITY;
#pragma unroll
        for (int n = 0; n < 2; ++n)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const int key = kb + n * 8 + 2 * qd + j;
            const float x = key < nvalid ? sc[n][2 * hr + j] * c : -INFINITY;
            sc[n][2 * hr + j] = x;
            mx = fmaxf(mx, x);
          }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float m_new = fmaxf(m_run[hr], mx);  // finite: key kb is valid
        corr[hr] = fast_exp2(m_run[hr] - m_new);
        m_run[hr] = m_new;
        float ls = 0.f;
#pragma unroll
        for (int n = 0; n < 2; ++n)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const float pv = fast_exp2(sc[n][2 * hr + j] - m_new);
            sc[n][2 * hr + j] = pv;
            ls += pv;
          }
        l_run[hr] = l_run[hr] * corr[hr] + ls;
      }
      if (__any_sync(0xffffffffu, corr[0] != 1.f || corr[1] != 1.f)) {
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          o[n][0] *= corr[0];
          o[n][1] *= corr[0];
          o[n][2] *= corr[1];
          o[n][3] *= corr[1];
        }
      }
      // ---- P as bf16 value + bf16 residual (A fragments, keys along k)
      uint32_t ph[4], pl[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int n = i >> 1, e0 = (i & 1) * 2;
        const float x0 = sc[n][e0], x1 = sc[n][e0 + 1];
        ph[i] = pack_bf16(x0, x1);
        pl[i] = pack_bf16(x0 - bf16_lo(ph[i]), x1 - bf16_hi(ph[i]));
      }
      // A fragment order: a0 (row r0, keys 0-7), a1 (row r0+8, keys 0-7),
      // a2 (row r0, keys 8-15), a3 (row r0+8, keys 8-15)
      const uint32_t ah[4] = {ph[0], ph[1], ph[2], ph[3]};
      const uint32_t al[4] = {pl[0], pl[1], pl[2], pl[3]};
      // ---- O += P V
      {
        const int vrow = kb + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int vsel = lane >> 4;
#pragma unroll
        for (int jj = 0; jj < NT / 2; ++jj) {
          uint32_t bv[4];
          ldsm_x4_t(vst + sw_off(vrow, 2 * jj + vsel), bv);
          mma_16816(o[2 * jj], ah, bv[0], bv[1]);
          mma_16816(o[2 * jj], al, bv[0], bv[1]);
          mma_16816(o[2 * jj + 1], ah, bv[2], bv[3]);
          mma_16816(o[2 * jj + 1], al, bv[2], bv[3]);
        }
      }
    }
    // this stage's generic stores (the appended row, the cleared V rows)
    // before the TMA refills it through the async proxy
    if (t == fresh_tile || nvalid < kTile) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncthreads();  // stage s is free again
    if (tid == 0 && issued < ntiles) {
      issue(issued);
      ++issued;
    }
  }

  // tiles requested past the length (only ever among the first kStages):
  // their copies land before the ring is reused for the merge
  if (ok && tid == 0) {
    for (int t = ntiles; t < issued; ++t) {
      int dummy = 0;
      if (!tc::mbar_wait(&full[t % kStages], (uint32_t)((t / kStages) & 1), &dummy, status)) break;
    }
  }
  if (ok) __syncthreads();
  if (!ok) {
    if (tid == 0) {
      // drain the copies still in flight before the CTA exits
      int dummy = 0;
      for (int s = 0; s < kStages && s < issued; ++s) {
        const int last = issued - 1 - ((issued - 1 - s) % kStages);
        tc::mbar_wait(&full[s], (uint32_t)((last / kStages) & 1), &dummy, status);
      }
    }
    return;
  }

  // ---- merge the eight warps: O, m, l through shared memory (the ring is free)
#pragma unroll
  for (int hr = 0; hr < 2; ++hr) {
    l_run[hr] += __shfl_xor_sync(0xffffffffu, l_run[hr], 1);
    l_run[hr] += __shfl_xor_sync(0xffffffffu, l_run[hr], 2);
  }
  constexpr int DS = Gm::kDS;
  float* mo = reinterpret_cast<float*>(smem);                // [kWarps][16][DS]
  float* mml = reinterpret_cast<float*>(smem + Gm::kMergeO);  // [kWarps][16][2]
  // only the G real query rows of the 16-row MMA tile are kept
  if (r0 < G) {
#pragma unroll
    for (int n = 0; n < NT; ++n)
      *reinterpret_cast<float2*>(mo + (warp * 16 + r0) * DS + n * 8 + 2 * qd) =
          make_float2(o[n][0], o[n][1]);
  }
  if (r0 + 8 < G) {
#pragma unroll
    for (int n = 0; n < NT; ++n)
      *reinterpret_cast<float2*>(mo + (warp * 16 + r0 + 8) * DS + n * 8 + 2 * qd) =
          make_float2(o[n][2], o[n][3]);
  }
  if (qd == 0) {
    mml[(warp * 16 + r0) * 2] = m_run[0];
    mml[(warp * 16 + r0) * 2 + 1] = l_run[0];
    mml[(warp * 16 + r0 + 8) * 2] = m_run[1];
    mml[(warp * 16 + r0 + 8) * 2 + 1] = l_run[1];
  }
  __syncthreads();
  // per head: the warps' weights 2^(m_w - M) (thread h), then every output
  // element as one pass of independent loads over the warps
  float* wgt = mml + kWarps * 16 * 2;  // [G][kWarps]
  if (tid < G) {
    const int h = tid;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, mml[(w * 16 + h) * 2]);
    float L = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float mw = mml[(w * 16 + h) * 2];
      const float wt = (M != -INFINITY && mw != -INFINITY) ? fast_exp2(mw - M) : 0.f;
      wgt[h * kWarps + w] = wt;
      L = fmaf(mml[(w * 16 + h) * 2 + 1], wt, L);
    }
    part_ml[part_base + (size_t)h * p.splits] = make_float2(M, L);
  }
  __syncthreads();
  for (int e = tid; e < G * (D / 4); e += kThreads) {
    const int h = e / (D / 4), d4 = e % (D / 4);
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float wt = wgt[h * kWarps + w];
      const float4 ow = *reinterpret_cast<const float4*>(mo + (w * 16 + h) * DS + 4 * d4);
      O.x = fmaf(ow.x, wt, O.x);
      O.y = fmaf(ow.y, wt, O.y);
      O.z = fmaf(ow.z, wt, O.z);
      O.w = fmaf(ow.w, wt, O.w);
    }
    *reinterpret_cast<float4*>(part_o + (part_base + (size_t)h * p.splits) * D + 4 * d4) = O;
  }

  // ---- with the merge kernel behind this one, the partials are all it leaves
  if (p.merge_kernel) return;
  // ---- otherwise the last split CTA of this (request, KV head) merges every split.
  // One thread counts the CTA in with an acquire-release atomic: the barrier
  // orders every thread's partial stores before it, the release makes them
  // visible with the count, and the last CTA's acquire (then its barrier)
  // orders its loads of the other splits' partials after it.
  __syncthreads();
  if (tid == 0) {
    int prev;
    asm volatile("atom.add.acq_rel.gpu.global.s32 %0, [%1], 1;"
                 : "=r"(prev)
                 : "l"(counters + b * p.hkv + g)
                 : "memory");
    *last_flag = prev == p.splits - 1;
    // every split has counted in: the counter goes back to zero for the next
    // call (what a prepared workspace relies on; the clearing kernel of the
    // other entry points zeroes it anyway)
    if (*last_flag) counters[b * p.hkv + g] = 0;
  }
  __syncthreads();
  if (!*last_flag) return;
  merge_splits<D, G, 1>(p, b, g, 0, part_o, part_ml, out, status, reinterpret_cast<float*>(smem), len);
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tma(const __grid_constant__ DecodeParams p, const __grid_constant__ CUtensorMap tk,
               const __grid_constant__ CUtensorMap tv, const uint16_t* __restrict__ kc,
               const uint16_t* __restrict__ vc, const uint16_t* __restrict__ q,
               const int32_t* __restrict__ lens, float* __restrict__ part_o,
               float2* __restrict__ part_ml, int32_t* __restrict__ counters,
               void* __restrict__ out, int32_t* __restrict__ status) {
  decode_tma_body<D, G>(p, tk, tv, kc, vc, q, lens, part_o, part_ml, counters, out, status);
  // Mode 3 never waited for the preceding kernel: one thread waits for it
  // now, after all of this CTA's work, so that this grid completes only after
  // that kernel has. Whatever waits for this grid (the merge kernel, the next
  // kernel's own dependency wait, the stream) then waits for both. The
  // preceding kernel's CTAs are all resident by now (it let this grid launch
  // only once every one of them had started), so the wait ends.
  if (p.early_tma == 3 && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 && threadIdx.x == 0)
    pdl_wait();
}

// The split merge as a kernel of its own, kMergeParts CTAs per (KV head,
// request), each on a quarter of the head dims (so that the splits' partial
// outputs are read by several SMs at once), launched behind the split kernel
// (programmatic dependent launch: resident while the split CTAs run, it waits
// for their completion), so that no split CTA waits on a split counter's
// round trip.
template <int D, int G>
__global__ void __launch_bounds__(kThreads) decode_merge(
    const __grid_constant__ DecodeParams p, const int32_t* __restrict__ lens,
    const float* __restrict__ part_o, const float2* __restrict__ part_ml, void* __restrict__ out,
    int32_t* __restrict__ status) {
  extern __shared__ float wts[];  // [G][splits]
  const int g = blockIdx.x, b = blockIdx.y, dpart = blockIdx.z;
  pdl_wait();
  pdl_trigger();
  const int64_t cap64 = p.max_len < (int64_t)p.cache_cap[b] ? p.max_len : (int64_t)p.cache_cap[b];
  int len = lens[b];
  if (len > (int)cap64) len = (int)cap64;  // (the split kernel flags it)
  if (len < 0) len = 0;
  merge_splits<D, G, kMergeParts>(p, b, g, dpart, part_o, part_ml, out, status, wts, len);
}

template <int D, int G>
cudaError_t launch_g(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                     const void* Kc, const void* Vc, const void* q, const int32_t* lens, float* part_o, float2* part_ml,
                     int32_t* counters, void* out, int32_t* status, cudaStream_t s) {
  using Gm = DGeo<D>;
  auto kern = decode_tma<D, G>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3(p.splits, p.hkv, p.batch), dim3(kThreads), Gm::kSmem, s, p, tk, tv,
                 static_cast<const uint16_t*>(Kc), static_cast<const uint16_t*>(Vc),
                 static_cast<const uint16_t*>(q), lens, part_o, part_ml, counters, out, status);
  if (e != cudaSuccess) return e;
  if (p.merge_kernel) {
    auto mk = decode_merge<D, G>;
    const size_t msmem = sizeof(float) * (size_t)G * p.splits;
    e = cudaFuncSetAttribute(mk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)msmem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(mk, dim3(p.hkv, p.batch, kMergeParts), dim3(kThreads), msmem, s, p, lens,
                   static_cast<const float*>(part_o), static_cast<const float2*>(part_ml), out, status);
    count_launches(1);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                     const void* Kc, const void* Vc, const void* q, const int32_t* lens, float* part_o, float2* part_ml,
                     int32_t* counters, void* out, int32_t* status, cudaStream_t s) {
  switch (p.group) {
#define TB_CASE(GG) \
  case GG:          \
    return launch_g<D, GG>(p, tk, tv, Kc, Vc, q, lens, part_o, part_ml, counters, out, status, s);
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
  const bool g_ok = (g >= 1 && g <= 8) || g == 12 || g == 16;  // rows of one 16-row MMA tile
  const int max_splits = p.d == 64 ? DGeo<64>::kMaxSplits : DGeo<128>::kMaxSplits;
  return p.dtype == TB_BF16 && (p.d == 64 || p.d == 128) && g_ok && p.splits <= max_splits &&
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
      p.d == 64 ? launch_d<64>(p, tk, tv, Kc, Vc, q, lens, part_o, part_ml, counters, out, status, s)
                : launch_d<128>(p, tk, tv, Kc, Vc, q, lens, part_o, part_ml, counters, out, status, s);
  count_launches(1);
  return e;
}

}  // namespace tb
