// Observation-window scoring on the sm_103a tensor cores (bf16 inputs).
//
// The same computation as the SIMT path (k_scores_simt.cu): for request b,
// KV head g and prefix key j,
//   S[g][j] = sum_{h in g, w < W} 2^(t_hwj - c_hw),   t = log2(e) q.k / sqrt(d),
// with c_hw the log2-sum-exp of window row (h, w) over the keys it sees
// (j <= P + w). The G*W <= 256 window rows of a group form one operand; the
// key tiles stream through shared memory by TMA and meet it in tcgen05.mma
// (bf16 x bf16 -> fp32 in TMEM). Two passes, because every row needs its
// global log-sum-exp before any key's score can be summed:
//
//  pass 1 (ws_stats_tc)  D[row][key] = Q K^T: each epilogue thread owns one
//                        window row and folds its keys into a running
//                        (max, sum of 2^(t - max)) pair;
//  pass 2 (ws_scores_tc) D[key][row] = K Q^T: each epilogue thread owns one
//                        key and sums 2^(t - c_row) over the rows, reading
//                        the key tiles in reverse order so that the tail the
//                        first pass loaded last is still in L2.
//
// Warp roles (640 threads, one CTA per SM): warp 0 issues TMA loads, warp 1
// issues the MMAs (one elected thread), warp 2 owns the TMEM allocation, and
// warps 4..19 are the epilogue: four per TMEM lane quadrant, each taking a
// quarter of the accumulator columns (the epilogue is latency-bound, so it
// wants many warps). Shared memory holds the
// window rows once and a 4-stage ring of key tiles; TMEM holds two 256-column
// accumulators so the MMA of tile t+1 overlaps the epilogue of tile t.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>

#include <mutex>

#include "tb_internal.cuh"
#include "tc_ptx.cuh"

namespace tb {
namespace {

constexpr int kTileKeys = 128;
constexpr int kStages = 4;
constexpr int kThreads = 640;
constexpr int kEpiWarp0 = 4;
constexpr int kEpiWarps = 16;  // four per TMEM lane quadrant, each on a quarter of the columns
constexpr uint32_t kTmemCols = 512;
constexpr int kBoxBytes = 128 * 128;  // one TMA box: 128 rows x 64 bf16
// Of every 32 exponentials an epilogue thread takes, the first kMufuElems go
// to the MUFU unit and the rest to the FMA pipes (tc::exp2_poly2). Measured on
// GB300: sending 12 of 32 to the FMA pipes slowed both passes (the epilogue is
// bound by latency, not by MUFU throughput), so all of them use MUFU.
constexpr int kMufuElems = 32;

template <int D>
struct Geo {
  static constexpr int KH = D / 64;                  // 64-column k-halves
  static constexpr int kQHalf = 256 * 128;           // 256 window rows x 128 B
  static constexpr int kQBytes = KH * kQHalf;
  static constexpr int kTileBytes = KH * kBoxBytes;  // 128 keys x D bf16
  static constexpr int kKSteps = D / 16;
  static constexpr int kRingOff = kQBytes;
  static constexpr int kBarOff = kRingOff + kStages * kTileBytes;
  static constexpr int kCrOff = kBarOff + 1024;
  static constexpr int kXOff = kCrOff + 256 * 4;       // pass 2: 2 x 3 x 128 partial sums
  static constexpr int kMOff = kXOff + 2 * 3 * 128 * 4;  // pass 1: 256 (max, sum) pairs
  static constexpr int kSmem = kMOff + 256 * 8 + 1024;   // + alignment slack
};

struct Bars {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t qfull;
  uint64_t xfull[2];   // pass 2: the second warpgroup's half sums are in xbuf
  uint64_t xempty[2];  // pass 2: the first warpgroup consumed them
  uint32_t tmem_base;
  int abort;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

struct ItemInfo {
  int b, g, j0, j1;
};

__device__ __forceinline__ ItemInfo locate(const EvictParams& p, int item, bool prefix_only) {
  int b = 0;
  while (b + 1 < p.batch && p.req[b + 1].item0 <= item) ++b;
  const EvictReq& rq = p.req[b];
  const int nch = (rq.n + p.chunk - 1) / p.chunk;
  const int local = item - rq.item0;
  ItemInfo it;
  it.b = b;
  it.g = local / nch;
  it.j0 = (local % nch) * p.chunk;
  it.j1 = min(prefix_only ? rq.p : rq.n, it.j0 + p.chunk);
  return it;
}

// Common set-up: barriers and the TMEM allocation. Returns the TMEM base.
__device__ __forceinline__ uint32_t setup(Bars* bars) {
  const int warp = threadIdx.x / 32;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&bars->full[s], 1);
      tc::mbar_init(&bars->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      tc::mbar_init(&bars->tfull[a], 1);
      tc::mbar_init(&bars->tempty[a], kEpiWarps);
    }
    tc::mbar_init(&bars->qfull, 1);
    for (int x = 0; x < 2; ++x) {
      tc::mbar_init(&bars->xfull[x], kEpiWarps * 3 / 4);
      tc::mbar_init(&bars->xempty[x], kEpiWarps / 4);
    }
    bars->abort = 0;
    tc::fence_barrier_init();
  }
  if (warp == 2) tc::tmem_alloc(&bars->tmem_base, kTmemCols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  return bars->tmem_base;
}

// Producer and MMA drains + TMEM release, run by every thread at the end.
__device__ __forceinline__ void teardown(Bars* bars, uint32_t tmem, int issued, int committed,
                                         int32_t* status) {
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  volatile int* abort = &bars->abort;
  if (warp == 0 && lane == 0 && *abort) {
    // wait for the copies still in flight so no copy lands after exit
    int dummy = 0;
    tc::mbar_wait(&bars->qfull, 0, &dummy, status);
    for (int s = 0; s < kStages && s < issued; ++s) {
      const int last = issued - 1 - ((issued - 1 - s) % kStages);
      int dummy = 0;
      tc::mbar_wait(&bars->full[s], (uint32_t)((last / kStages) & 1), &dummy, status);
    }
  }
  if (warp == 1 && lane == 0 && committed > 0) {
    // the last accumulator commit covers every MMA this thread issued
    const int last = committed - 1;
    int dummy = 0;
    tc::mbar_wait(&bars->tfull[last & 1], (uint32_t)((last >> 1) & 1), &dummy, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// pass 1: per-row (max, sum) over one chunk of keys
// ---------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    ws_stats_tc(const __grid_constant__ EvictParams p, const __grid_constant__ CUtensorMap tq,
                const __grid_constant__ CUtensorMap tk, float2* __restrict__ partial,
                int32_t* __restrict__ status) {
  using G = Geo<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* q_s = smem;
  uint8_t* ring = smem + G::kRingOff;
  Bars* bars = reinterpret_cast<Bars*>(smem + G::kBarOff);
  float2* mrg = reinterpret_cast<float2*>(smem + G::kMOff);
  bool my_ok = false;
  float my_m = -INFINITY, my_l = 0.f;

  const int item = blockIdx.x;
  const ItemInfo info = locate(p, item, false);
  const EvictReq& rq = p.req[info.b];
  const int ntiles = (info.j1 - info.j0 + kTileKeys - 1) / kTileKeys;
  const int M = p.m_rows;
  const int RB = M > 128 ? 2 : 1;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t tmem = setup(bars);
  volatile int* abort = &bars->abort;
  int issued = 0, committed = 0;

  if (warp == 0) {
    if (lane == 0) {
      tc::tma_prefetch_desc(&tq);
      tc::tma_prefetch_desc(&tk);
      const int qrow = (info.b * p.hq + info.g * p.group) * p.window;
      tc::mbar_arrive_expect_tx(&bars->qfull, (uint32_t)(RB * G::KH * kBoxBytes));
      for (int h = 0; h < G::KH; ++h)
        for (int rb = 0; rb < RB; ++rb)
          tc::tma_load_2d(q_s + h * G::kQHalf + rb * kBoxBytes, &tq, h * 64, qrow + rb * 128,
                          &bars->qfull);
      const int krow = (int)((int64_t)info.g * p.kv_rows + rq.kv_off) + info.j0;
      for (int it = 0; it < ntiles; ++it) {
        const int s = it % kStages;
        if (!tc::mbar_wait(&bars->empty[s], ((it / kStages) & 1) ^ 1, abort, status)) break;
        tc::mbar_arrive_expect_tx(&bars->full[s], (uint32_t)G::kTileBytes);
        for (int h = 0; h < G::KH; ++h)
          tc::tma_load_2d(ring + s * G::kTileBytes + h * kBoxBytes, &tk, h * 64,
                          krow + it * kTileKeys, &bars->full[s]);
        issued = it + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && tc::mbar_wait(&bars->qfull, 0, abort, status)) {
      constexpr uint32_t idesc = tc::idesc_bf16(128, kTileKeys);
      for (int it = 0; it < ntiles; ++it) {
        const int s = it % kStages, a = it & 1;
        if (!tc::mbar_wait(&bars->full[s], (it / kStages) & 1, abort, status)) break;
        if (!tc::mbar_wait(&bars->tempty[a], ((it >> 1) & 1) ^ 1, abort, status)) break;
        tc::tc_fence_after();
        const uint32_t kbase = tc::smem_addr(ring + s * G::kTileBytes);
        const uint32_t qbase = tc::smem_addr(q_s);
#pragma unroll
        for (int kk = 0; kk < G::kKSteps; ++kk) {
          const uint32_t off = (uint32_t)((kk >> 2) * kBoxBytes + (kk & 3) * 32);
          const uint64_t bdesc = tc::sw128_desc(kbase + off);
          for (int rb = 0; rb < RB; ++rb) {
            const uint64_t adesc =
                tc::sw128_desc(qbase + (uint32_t)((kk >> 2) * G::kQHalf + rb * kBoxBytes + (kk & 3) * 32));
            tc::mma_bf16(tmem + (uint32_t)(a * 256 + rb * 128), adesc, bdesc, idesc, kk > 0);
          }
        }
        tc::mma_commit(&bars->empty[s]);
        tc::mma_commit(&bars->tfull[a]);
        committed = it + 1;
      }
    }
  } else if (warp >= kEpiWarp0) {
    // rows: row block wg, TMEM lane quadrant quad; columns: half `half` of the tile
    const int e = warp - kEpiWarp0, sub = e >> 2, quad = warp & 3;
    const int wg = sub >> 1, half = sub & 1;
    const int row = wg * 128 + quad * 32 + lane;
    const int w = row % p.window;
    const int vis_end = min(rq.n, rq.p + w + 1);  // keys [0, vis_end) visible to the row
    const float c = p.scale_log2;
    float m_run = -INFINITY;
    float l_run = 0.f, l_comp = 0.f;  // compensated running sum of 2^(t - m_run)
    bool ok = true;
    for (int it = 0; it < ntiles; ++it) {
      const int a = it & 1;
      if (!tc::mbar_wait(&bars->tfull[a], (it >> 1) & 1, abort, status)) {
        ok = false;
        break;
      }
      tc::tc_fence_after();
      if (wg < RB) {
        const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(a * 256 + wg * 128);
        const int key0 = info.j0 + it * kTileKeys;
        const bool all_vis = key0 + kTileKeys <= rq.p;
#pragma unroll 1
        for (int ch = 2 * half; ch < 2 * half + 2; ++ch) {
          float v[32];
          __syncwarp();
          tc::tmem_ld32(taddr + ch * 32, v);
          tc::tmem_ld_wait();
          if (!all_vis) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (key0 + ch * 32 + i >= vis_end) v[i] = -INFINITY;
          }
          // chunk max with three-input max (tree of 16 + 5 + 2 + 1 ops)
          float mt[11];
#pragma unroll
          for (int i = 0; i < 10; ++i) mt[i] = tc::max3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
          mt[10] = fmaxf(v[30], v[31]);
          const float mx = tc::max3(tc::max3(mt[0], mt[1], mt[2]), tc::max3(mt[3], mt[4], mt[5]),
                                    tc::max3(tc::max3(mt[6], mt[7], mt[8]), mt[9], mt[10]));
          const float m_new = fmaxf(m_run, mx * c);
          if (m_new != -INFINITY) {  // some key of this chunk is visible
            if (m_new > m_run) {
              const float sc = fast_exp2(m_run - m_new);
              l_run *= sc;
              l_comp *= sc;
              m_run = m_new;
            }
            // 2^(v c - m) in packed pairs, summed in two packed accumulators
            const uint64_t cc = tc::pk2(c, c), mm = tc::pk2(-m_run, -m_run);
            uint64_t acc0 = 0, acc1 = 0;
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              const float2 a = tc::upk2(tc::fma2(tc::pk2(v[i], v[i + 1]), cc, mm));
              const float2 bq = tc::upk2(tc::fma2(tc::pk2(v[i + 2], v[i + 3]), cc, mm));
              float2 ea, eb;
              if (i < kMufuElems) {
                ea = make_float2(fast_exp2(a.x), fast_exp2(a.y));
                eb = make_float2(fast_exp2(bq.x), fast_exp2(bq.y));
              } else {
                ea = tc::exp2_poly2(a.x, a.y);
                eb = tc::exp2_poly2(bq.x, bq.y);
              }
              acc0 = tc::add2(acc0, tc::pk2(ea.x, ea.y));
              acc1 = tc::add2(acc1, tc::pk2(eb.x, eb.y));
            }
            const float2 s01 = tc::upk2(tc::add2(acc0, acc1));
            const float term = (s01.x + s01.y) - l_comp;
            const float tsum = l_run + term;
            l_comp = (tsum - l_run) - term;
            l_run = tsum;
          }
        }
      }
      tc::tc_fence_before();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->tempty[a]);
    }
    // the second column half hands its (max, sum) to the first
    if (half == 1) mrg[row] = make_float2(ok ? m_run : NAN, l_run);
    my_ok = ok;
    my_m = m_run;
    my_l = l_run;
  }
  __syncthreads();
  if (warp >= kEpiWarp0) {
    const int e = warp - kEpiWarp0, sub = e >> 2, quad = warp & 3;
    const int wg = sub >> 1, half = sub & 1;
    const int row = wg * 128 + quad * 32 + lane;
    if (half == 0 && wg < RB && row < M) {
      const float2 o = mrg[row];
      if (my_ok && !isnan(o.x)) {
        const float m = fmaxf(my_m, o.x);
        const float l = (m == -INFINITY) ? 0.f
                                        : my_l * fast_exp2(my_m - m) + o.y * fast_exp2(o.x - m);
        partial[(size_t)item * M + row] = make_float2(m, l);
      }
    }
  }
  teardown(bars, tmem, issued, committed, status);
}

// ---------------------------------------------------------------------------
// pass 2: per-key normalised window sum
// ---------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    ws_scores_tc(const __grid_constant__ EvictParams p, const __grid_constant__ CUtensorMap tq,
                 const __grid_constant__ CUtensorMap tk, const float* __restrict__ rowc,
                 float* __restrict__ scores, int32_t* __restrict__ status) {
  using G = Geo<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* q_s = smem;
  uint8_t* ring = smem + G::kRingOff;
  Bars* bars = reinterpret_cast<Bars*>(smem + G::kBarOff);
  float* cr = reinterpret_cast<float*>(smem + G::kCrOff);
  float* xbuf = reinterpret_cast<float*>(smem + G::kXOff);

  const int item = blockIdx.x;
  const ItemInfo info = locate(p, item, true);
  if (info.j1 <= info.j0) return;  // this chunk holds window keys only
  const EvictReq& rq = p.req[info.b];
  const int ntiles = (info.j1 - info.j0 + kTileKeys - 1) / kTileKeys;
  const int M = p.m_rows;
  const int NP = (M + 15) & ~15;  // MMA N: window rows rounded up to 16
  const int RBQ = NP > 128 ? 2 : 1;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  const float* rc = rowc + ((size_t)info.b * p.hkv + info.g) * M;
  float* ncr = cr;  // -c_row; -inf for padding rows so that their terms vanish
  for (int r = threadIdx.x; r < 256; r += blockDim.x) ncr[r] = r < M ? -rc[r] : -INFINITY;
  const uint32_t tmem = setup(bars);
  volatile int* abort = &bars->abort;
  int issued = 0, committed = 0;

  if (warp == 0) {
    if (lane == 0) {
      tc::tma_prefetch_desc(&tq);
      tc::tma_prefetch_desc(&tk);
      const int qrow = (info.b * p.hq + info.g * p.group) * p.window;
      tc::mbar_arrive_expect_tx(&bars->qfull, (uint32_t)(RBQ * G::KH * kBoxBytes));
      for (int h = 0; h < G::KH; ++h)
        for (int rb = 0; rb < RBQ; ++rb)
          tc::tma_load_2d(q_s + h * G::kQHalf + rb * kBoxBytes, &tq, h * 64, qrow + rb * 128,
                          &bars->qfull);
      const int krow = (int)((int64_t)info.g * p.kv_rows + rq.kv_off) + info.j0;
      for (int it = 0; it < ntiles; ++it) {
        const int s = it % kStages;
        const int t = ntiles - 1 - it;  // reverse order: the first pass's tail is in L2
        if (!tc::mbar_wait(&bars->empty[s], ((it / kStages) & 1) ^ 1, abort, status)) break;
        tc::mbar_arrive_expect_tx(&bars->full[s], (uint32_t)G::kTileBytes);
        for (int h = 0; h < G::KH; ++h)
          tc::tma_load_2d(ring + s * G::kTileBytes + h * kBoxBytes, &tk, h * 64,
                          krow + t * kTileKeys, &bars->full[s]);
        issued = it + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && tc::mbar_wait(&bars->qfull, 0, abort, status)) {
      const uint32_t idesc = tc::idesc_bf16(128, NP);
      for (int it = 0; it < ntiles; ++it) {
        const int s = it % kStages, a = it & 1;
        if (!tc::mbar_wait(&bars->full[s], (it / kStages) & 1, abort, status)) break;
        if (!tc::mbar_wait(&bars->tempty[a], ((it >> 1) & 1) ^ 1, abort, status)) break;
        tc::tc_fence_after();
        const uint32_t kbase = tc::smem_addr(ring + s * G::kTileBytes);
        const uint32_t qbase = tc::smem_addr(q_s);
#pragma unroll
        for (int kk = 0; kk < G::kKSteps; ++kk) {
          const uint64_t adesc = tc::sw128_desc(kbase + (uint32_t)((kk >> 2) * kBoxBytes + (kk & 3) * 32));
          const uint64_t bdesc = tc::sw128_desc(qbase + (uint32_t)((kk >> 2) * G::kQHalf + (kk & 3) * 32));
          tc::mma_bf16(tmem + (uint32_t)(a * 256), adesc, bdesc, idesc, kk > 0);
        }
        tc::mma_commit(&bars->empty[s]);
        tc::mma_commit(&bars->tfull[a]);
        committed = it + 1;
      }
    }
  } else if (warp >= kEpiWarp0) {
    // keys: TMEM lane quadrant quad; window rows (columns): quarter `sub`
    const int e = warp - kEpiWarp0, sub = e >> 2, quad = warp & 3;
    const int key = quad * 32 + lane;  // TMEM lane = key within the tile
    const float c = p.scale_log2;
    float* out = scores + (size_t)info.g * p.score_rows + rq.score_off;
    for (int it = 0; it < ntiles; ++it) {
      const int a = it & 1;
      const int t = ntiles - 1 - it;
      if (!tc::mbar_wait(&bars->tfull[a], (it >> 1) & 1, abort, status)) break;
      tc::tc_fence_after();
      const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(a * 256);
      float acc = 0.f;
#pragma unroll 1
      for (int ch = 0; ch < 2; ++ch) {
        const int c0 = sub * 64 + ch * 32;
        if (c0 >= NP) break;
        float v[32];
        __syncwarp();
        tc::tmem_ld32(taddr + c0, v);
        tc::tmem_ld_wait();
        // 2^(v c - c_row) in packed pairs; -c_row pairs come from shared memory
        const uint64_t c2 = tc::pk2(c, c);
        uint64_t a0 = 0, a1 = 0;
#pragma unroll
        for (int i = 0; i < 32; i += 4) {
          const float4 nc = *reinterpret_cast<const float4*>(ncr + c0 + i);
          const float2 x = tc::upk2(tc::fma2(tc::pk2(v[i], v[i + 1]), c2, tc::pk2(nc.x, nc.y)));
          const float2 y = tc::upk2(tc::fma2(tc::pk2(v[i + 2], v[i + 3]), c2, tc::pk2(nc.z, nc.w)));
          float2 ex, ey;
          if (i < kMufuElems) {
            ex = make_float2(fast_exp2(x.x), fast_exp2(x.y));
            ey = make_float2(fast_exp2(y.x), fast_exp2(y.y));
          } else {
            ex = tc::exp2_poly2(x.x, x.y);
            ey = tc::exp2_poly2(y.x, y.y);
          }
          a0 = tc::add2(a0, tc::pk2(ex.x, ex.y));
          a1 = tc::add2(a1, tc::pk2(ey.x, ey.y));
        }
        const float2 s01 = tc::upk2(tc::add2(a0, a1));
        acc += s01.x + s01.y;
      }
      tc::tc_fence_before();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->tempty[a]);
      // combine the four quarters of the window rows through a double-buffered
      // hand-off (bounded mbarrier waits, no named barrier); fixed sum order
      const int x = it & 1;
      const uint32_t xph = (uint32_t)((it >> 1) & 1);
      if (sub > 0) {
        if (!tc::mbar_wait(&bars->xempty[x], xph ^ 1, abort, status)) break;
        xbuf[(x * 3 + sub - 1) * 128 + key] = acc;
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->xfull[x]);
      } else {
        if (!tc::mbar_wait(&bars->xfull[x], xph, abort, status)) break;
        const int j = info.j0 + t * kTileKeys + key;
        const float* xb = xbuf + x * 3 * 128;
        if (j < info.j1) out[j] = ((acc + xb[key]) + xb[128 + key]) + xb[256 + key];
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->xempty[x]);
      }
    }
  }
  teardown(bars, tmem, issued, committed, status);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

bool make_map(CUtensorMap* map, const void* base, int d, uint64_t rows) {
  return make_bf16_map(map, base, d, rows, 128);
}

}  // namespace

// 2-D bf16 map over rows of `d` elements: boxes of box_rows rows x 64
// columns, 128-byte swizzle (the layout the MMA descriptors expect).
bool make_bf16_map(CUtensorMap* map, const void* base, int d, uint64_t rows, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

template <int D>
cudaError_t launch_tc_typed(const EvictParams& pt, const CUtensorMap& tq, const CUtensorMap& tk,
                            float* scores, float2* partial, float* rowc, int32_t* status,
                            cudaStream_t s) {
  using Gm = Geo<D>;
  cudaError_t e = cudaFuncSetAttribute(ws_stats_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Gm::kSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(ws_scores_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  ws_stats_tc<D><<<pt.items, kThreads, Gm::kSmem, s>>>(pt, tq, tk, partial, status);
  launch_window_combine(pt, partial, rowc, s);
  ws_scores_tc<D><<<pt.items, kThreads, Gm::kSmem, s>>>(pt, tq, tk, rowc, scores, status);
  count_launches(2);
  return cudaGetLastError();
}

}  // namespace

bool window_scores_tc_supported(const EvictParams& p) {
  const uint64_t krows = (uint64_t)p.hkv * (uint64_t)p.kv_rows;
  const uint64_t qrows = (uint64_t)p.batch * p.hq * p.window;
  return p.dtype == TB_BF16 && (p.d == 64 || p.d == 128) && p.m_rows <= 256 &&
         krows < (1ull << 31) && qrows < (1ull << 31) && encode_fn() != nullptr;
}

// Work items: each CTA takes `chunk` consecutive keys of one (request, KV
// head), sized so that about one CTA per SM of a 152-SM GB300 runs.
EvictParams tc_item_params(const EvictParams& p) {
  EvictParams pt = p;
  int64_t tiles = 0;
  for (int b = 0; b < p.batch; ++b) tiles += (int64_t)p.hkv * ((p.req[b].n + kTileKeys - 1) / kTileKeys);
  int64_t per_item = (tiles + 151) / 152;
  if (per_item < 2) per_item = 2;  // >= the SIMT chunk, so the workspace stays large enough
  pt.chunk = (int32_t)(per_item * kTileKeys);
  int64_t items = 0;
  for (int b = 0; b < p.batch; ++b) {
    pt.req[b].item0 = (int32_t)items;
    items += (int64_t)p.hkv * ((p.req[b].n + pt.chunk - 1) / pt.chunk);
  }
  pt.items = (int32_t)items;
  return pt;
}

cudaError_t launch_window_scores_tc(const EvictParams& p, const void* q_win, const void* K,
                                    float* scores, float2* partial, float* rowc, int32_t* status,
                                    cudaStream_t s) {
  const EvictParams pt = tc_item_params(p);
  CUtensorMap tq, tk;
  const uint64_t qrows = (uint64_t)p.batch * p.hq * p.window;
  const uint64_t krows = (uint64_t)p.hkv * p.kv_rows;
  if (!make_map(&tq, q_win, p.d, qrows) || !make_map(&tk, K, p.d, krows))
    return cudaErrorInvalidValue;
  return p.d == 64 ? launch_tc_typed<64>(pt, tq, tk, scores, partial, rowc, status, s)
                   : launch_tc_typed<128>(pt, tq, tk, scores, partial, rowc, status, s);
}

}  // namespace tb
