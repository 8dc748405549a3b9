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
//  pass 1 (statistics)  D[row][key] = Q K^T: each epilogue thread owns one
//                       window row (and half of each tile's keys) and folds
//                       them into a running (max, sum of 2^(t - max)) pair;
//  pass 2 (votes)       D[key][row] = K Q^T: each epilogue thread owns one key
//                       (and a quarter of the rows) and sums 2^(t - c_row),
//                       reading the key tiles in reverse order so that the
//                       tail pass 1 loaded last is still in L2. The four
//                       quarter sums of a key meet in global memory: the launch
//                       that runs pass 1 clears the scores first (for the
//                       votes-only launch fed by the prefill's log-sum-exp, the
//                       caller's clearing kernel does), and each warp adds its
//                       sum with a reduction (no hand-off between the warps of
//                       a lane quadrant).
//
// One kernel template runs pass 1, pass 2, or both. Both (the default) is a
// cooperative launch of one CTA per SM: after pass 1 every CTA publishes its
// per-row partials, meets the others at a grid barrier (bounded wait), and
// merges the partials of its own KV head into c_row itself; meanwhile its TMA
// and MMA warps have already moved on to pass 2's first tiles. The fallback,
// when the grid cannot be co-resident, is pass 1, a merge kernel, then pass 2.
//
// Warp roles (576 threads, one CTA per SM): warps 0..15 are the epilogue, four
// per TMEM lane quadrant, each taking a quarter of the accumulator columns
// (the epilogue is latency-bound, so it wants many warps); warp 16 issues TMA
// loads and owns the TMEM allocation; warp 17 issues the MMAs (one elected
// lane of the converged warp).
// Shared memory holds the window rows once and a 4-stage ring of key tiles;
// TMEM holds two 256-column accumulators so the MMA of tile t+1 overlaps the
// epilogue of tile t.
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
constexpr int kThreads = 576;
constexpr int kEpiWarps = 16;      // four per TMEM lane quadrant
constexpr int kProducerWarp = 16;  // TMA issue; also owns the TMEM allocation
constexpr int kMmaWarp = 17;       // tcgen05.mma issue
constexpr uint32_t kTmemCols = 512;
constexpr int kBoxBytes = 128 * 128;  // one TMA box: 128 rows x 64 bf16
// Set in the grid-barrier word when a row maximum is too large for the fp64
// row sums (those heads then merge their partials the slow way).
constexpr uint32_t kSumOverflowBit = 0x80000000u;
// When some head is scored by more CTAs than this, the fused kernel sums its
// rows' (max, sum) partials in fp64 atomically as pass 1 ends (the kRowSums
// instantiation), so that after the grid barrier c_row is one load per row
// instead of a merge over every chunk. Measured on GB300: with 37 chunks per
// head (32K) the scoring took 26.4 -> 24.2 us; with 19 (128K) it did not pay.
constexpr int kSumMinChunks = 24;

// kRowSums (with kPassBoth): the fp64 row sums replace the post-barrier
// merge; a separate instantiation, so the kernel without it is unchanged
// kRedVotes: the launch that runs pass 1 zeroes the scores as it starts, and
// pass 2's warps add their quarter sums of the window rows into them with
// global reductions (no hand-off between the four warps of a lane quadrant).
// Every launch that runs pass 2 carries it (the votes-only launch adds into
// scores its caller cleared). Measured on GB300 (128K, per call): against a
// shared-memory hand-off, 114.8 -> 108.7 us for both passes and 64.8 ->
// 59.1 us for the votes-only launch, with each warp's reduction issued after
// its next TMEM load wait and relaxed hand-back arrivals (issued before the
// wait, or behind a release arrival, the stores stalled the warp: 134 us).
enum : int { kPassStats = 1, kPassVotes = 2, kPassBoth = 3, kRowSums = 4, kRedVotes = 8 };

template <int D>
struct Geo {
  static constexpr int KH = D / 64;                  // 64-column k-halves
  static constexpr int kQHalf = 256 * 128;           // 256 window rows x 128 B
  static constexpr int kQBytes = KH * kQHalf;
  static constexpr int kTileBytes = KH * kBoxBytes;  // 128 keys x D bf16
  static constexpr int kKSteps = D / 16;
  static constexpr int kRingOff = kQBytes;
  static constexpr int kBarOff = kRingOff + kStages * kTileBytes;
  static constexpr int kCrOff = kBarOff + 1024;          // -c_row for 256 rows
  static constexpr int kMOff = kCrOff + 256 * 4;         // pass 1: 256 (max, sum) pairs
  static constexpr int kSmem = kMOff + 256 * 8 + 1024;   // + alignment slack
};

struct Bars {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t qfull;
  uint64_t mrg;       // pass 1: the second column halves wrote their (max, sum)
  uint64_t pub;       // both passes: the CTA's partials are written
  uint64_t gready;    // both passes: every CTA of the grid published
  uint64_t crdone;    // -c_row is in shared memory
  uint32_t tmem_base;
  int abort;
  int codes[8];   // tile code of the it-th tile the producer claimed, at [it % 8]
  int accode[2];  // the MMA warp's copy for the accumulator it fills
  int sums_ok;    // kRowSums: every row's fp64 sum is usable (no row max beyond the range)
};

// Tile codes: t >= 0 is pass 1 tile t, -2 - t is pass 2 tile t, kNoTile ends.
constexpr int kNoTile = -1;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

struct ItemInfo {
  int b, g;      // request, KV head
  int ch, nch;   // this CTA's index among the (request, KV head)'s CTAs, their count
};

__device__ __forceinline__ ItemInfo locate(const EvictParams& p, int item) {
  int b = 0;
  while (b + 1 < p.batch && p.req[b + 1].item0 <= item) ++b;
  const EvictReq& rq = p.req[b];
  const int nch = (rq.n + p.chunk - 1) / p.chunk;
  const int local = item - rq.item0;
  ItemInfo it;
  it.b = b;
  it.g = local / nch;
  it.ch = local % nch;
  it.nch = nch;
  return it;
}

// Byte offset of k-step kk (16 bf16 = 32 B) inside a 128B-swizzled K-major
// operand made of 64-column boxes.
__host__ __device__ constexpr uint32_t kstep_off(int kk) {
  return (uint32_t)((kk >> 2) * kBoxBytes + (kk & 3) * 32);
}

// A shared-memory descriptor moved on by `bytes`: the start address field
// holds address >> 4 in the low 14 bits, and every operand here lies below
// 2^18 bytes, so the sum never carries out of the low word's field.
__device__ __forceinline__ uint64_t desc_plus(uint64_t d, uint32_t bytes) {
  return (d & 0xFFFFFFFF00000000ull) | (uint32_t)((uint32_t)d + (bytes >> 4));
}

// Pass 1 MMAs of k-steps [K0, K1) of one key tile, D[row][key] = Q K^T: one
// M=128 MMA per row block per k-step, all descriptors derived from two bases
// at compile-time offsets (the issue rate of these small MMAs bounds pass 1
// otherwise).
template <int D, int RB, int K0, int K1>
__device__ __forceinline__ void mma_stats_steps(uint32_t d_tmem, uint64_t qdesc, uint64_t kdesc,
                                                uint32_t on) {
  constexpr uint32_t idesc = tc::idesc_bf16(128, kTileKeys);
#pragma unroll
  for (int kk = K0; kk < K1; ++kk) {
    const uint64_t bdesc = desc_plus(kdesc, kstep_off(kk));
#pragma unroll
    for (int rb = 0; rb < RB; ++rb)
      tc::mma_bf16_if(d_tmem + (uint32_t)(rb * 128),
                      desc_plus(qdesc, (uint32_t)((kk >> 2) * Geo<D>::kQHalf + rb * kBoxBytes +
                                                  (kk & 3) * 32)),
                      bdesc, idesc, kk > 0, on);
  }
}

// Pass 2 MMAs of k-steps [K0, K1) of one key tile, D[key][row] = K Q^T over
// the window rows (N = their count rounded up to 16).
template <int D, int K0, int K1>
__device__ __forceinline__ void mma_votes_steps(uint32_t d_tmem, uint64_t qdesc, uint64_t kdesc,
                                                uint32_t idesc, uint32_t on) {
#pragma unroll
  for (int kk = K0; kk < K1; ++kk)
    tc::mma_bf16_if(d_tmem, desc_plus(kdesc, kstep_off(kk)),
                    desc_plus(qdesc, (uint32_t)((kk >> 2) * Geo<D>::kQHalf + (kk & 3) * 32)), idesc,
                    kk > 0, on);
}

template <int D, int K0, int K1>
__device__ __forceinline__ void mma_tile_steps(bool stats, int rb_count, uint32_t d_tmem,
                                               uint64_t qdesc, uint64_t kdesc, uint32_t idesc2,
                                               uint32_t on) {
  if (!stats)
    mma_votes_steps<D, K0, K1>(d_tmem, qdesc, kdesc, idesc2, on);
  else if (rb_count == 2)
    mma_stats_steps<D, 2, K0, K1>(d_tmem, qdesc, kdesc, on);
  else
    mma_stats_steps<D, 1, K0, K1>(d_tmem, qdesc, kdesc, on);
}

// sum over i < NV of 2^(v[i] c + bias[i]) in packed pairs, two packed
// accumulators; the biases (-c_row of each window row) come from shared memory
template <int NV>
__device__ __forceinline__ float vote_sum(const float (&v)[64], float c, const float* bias) {
  const uint64_t c2 = tc::pk2(c, c);
  uint64_t a0 = 0, a1 = 0;
#pragma unroll
  for (int i = 0; i < NV; i += 4) {
    const float4 nc = *reinterpret_cast<const float4*>(bias + i);
    const float2 x = tc::upk2(tc::fma2(tc::pk2(v[i], v[i + 1]), c2, tc::pk2(nc.x, nc.y)));
    const float2 y = tc::upk2(tc::fma2(tc::pk2(v[i + 2], v[i + 3]), c2, tc::pk2(nc.z, nc.w)));
    a0 = tc::add2(a0, tc::pk2(fast_exp2(x.x), fast_exp2(x.y)));
    a1 = tc::add2(a1, tc::pk2(fast_exp2(y.x), fast_exp2(y.y)));
  }
  const float2 s01 = tc::upk2(tc::add2(a0, a1));
  return s01.x + s01.y;
}

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    ws_tc(const __grid_constant__ EvictParams p, const __grid_constant__ CUtensorMap tq,
          const __grid_constant__ CUtensorMap tk, float2* __restrict__ partial,
          const float* __restrict__ rowc, float* __restrict__ scores, int32_t* __restrict__ status,
          uint32_t* __restrict__ gsync, int32_t* __restrict__ tilectr,
          double* __restrict__ lsum) {
  using G = Geo<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* q_s = smem;
  uint8_t* ring = smem + G::kRingOff;
  Bars* bars = reinterpret_cast<Bars*>(smem + G::kBarOff);
  float* ncr = reinterpret_cast<float*>(smem + G::kCrOff);
  float2* mrg = reinterpret_cast<float2*>(smem + G::kMOff);

  const int item = blockIdx.x;
  const ItemInfo info = locate(p, item);
  const EvictReq& rq = p.req[info.b];
  // Key tiles of this (request, KV head): pass 1 all N keys, pass 2 the P
  // prefix keys. Its CTAs claim them from two counters in the workspace, so
  // a CTA that runs slower takes fewer tiles (a static split left the grid
  // barrier waiting ~10 us for the slowest CTA).
  const int nt1 = (MODE & kPassStats) ? (rq.n + kTileKeys - 1) / kTileKeys : 0;
  const int nt2 = (MODE & kPassVotes) ? (rq.p + kTileKeys - 1) / kTileKeys : 0;
  if (nt1 + nt2 == 0) return;
  const int M = p.m_rows;
  const int RB = M > 128 ? 2 : 1;  // 128-row blocks of the window rows
  const int NP = (M + 15) & ~15;   // pass 2 MMA N: window rows rounded up to 16
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const size_t segrow = ((size_t)info.b * p.hkv + info.g) * M;
  constexpr bool kFused = (MODE & kPassBoth) == kPassBoth;
  constexpr bool kSums = kFused && (MODE & kRowSums) != 0;
  static_assert(!(MODE & kPassVotes) || (MODE & kRedVotes), "pass 2 adds by reductions");
  float* const sc_out = scores + (size_t)info.g * p.score_rows + rq.score_off;


  // ---- set-up: barriers and the TMEM allocation
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
    tc::mbar_init(&bars->mrg, kEpiWarps / 2);
    tc::mbar_init(&bars->pub, kEpiWarps);
    tc::mbar_init(&bars->gready, 1);
    tc::mbar_init(&bars->crdone, kEpiWarps);
    bars->abort = 0;
    tc::fence_barrier_init();
  }
  if (warp == kProducerWarp) tc::tmem_alloc(&bars->tmem_base, kTmemCols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  // global memory from here on (the votes-only launch is a programmatic
  // dependent launch: its set-up above overlapped the previous kernel)
  pdl_wait();
  if ((MODE & kRedVotes) && (MODE & kPassStats)) {
    // the launch that runs pass 1 clears every score before any pass 2 tile
    // adds into it (the grid barrier, or the launch boundary, orders the two);
    // these stores go out while the first key tiles are on their way
    const size_t total = (size_t)p.hkv * (size_t)p.score_rows;
    const size_t per = (total + gridDim.x - 1) / gridDim.x;
    const size_t z0 = per * blockIdx.x;
    const int cnt = z0 < total ? (int)min(per, total - z0) : 0;
    float* z = scores + z0;
    for (int i = threadIdx.x; i < cnt; i += blockDim.x) z[i] = 0.f;
  }
  if ((MODE & kPassBoth) == kPassVotes) {
    for (int r = threadIdx.x; r < 256; r += blockDim.x)
      ncr[r] = r < M ? -(rowc[segrow + r] * p.rowc_scale) : -INFINITY;
    debug_flag(threadIdx.x < M && !isfinite(ncr[threadIdx.x]), status);
    __syncthreads();
  }
  // (no early pdl_trigger here: the select's CTAs launched during the scoring
  // made the 128K step ~2 us slower on GB300; the select starts on completion)
  const uint32_t tmem = bars->tmem_base;
  volatile int* abort = &bars->abort;
  int issued = 0, committed = 0;

  if (warp == kProducerWarp) {
    // ---------------------------------------------------------------- TMA
    if (lane == 0) {
      tc::tma_prefetch_desc(&tq);
      tc::tma_prefetch_desc(&tk);
      const int qrow = (info.b * p.hq + info.g * p.group) * p.window;
      tc::mbar_arrive_expect_tx(&bars->qfull, (uint32_t)(RB * G::KH * kBoxBytes));
      for (int h = 0; h < G::KH; ++h)
        for (int rb = 0; rb < RB; ++rb)
          tc::tma_load_2d(q_s + h * G::kQHalf + rb * kBoxBytes, &tq, h * 64, qrow + rb * 128,
                          &bars->qfull);
      const int krow = (int)((int64_t)info.g * p.kv_rows + rq.kv_off);
      int* ctr = tilectr + 2 * (info.b * p.hkv + info.g);
      // pass 1 tiles in rising order, then pass 2 tiles from the top, so that
      // pass 2 starts on the tiles pass 1 loaded last (still in L2). A CTA's
      // first tile of each pass is its own index among the CTAs of the
      // (request, KV head); later claims count on from there, each issued one
      // tile ahead so that its round trip overlaps a wait.
      bool second = nt1 == 0;
      int claim = info.ch;
      for (int it = 0;; ++it) {
        const int s = it % kStages;
        if (!tc::mbar_wait(&bars->empty[s], ((it / kStages) & 1) ^ 1, abort, status)) break;
        if (!second && claim >= nt1) {
          // a stats-only launch leaves the pass 2 counter to the votes launch
          second = true;
          claim = nt2 > 0 ? info.ch : 0;
        }
        const int t = second ? (claim < nt2 ? nt2 - 1 - claim : -1) : claim;
        const int code = t < 0 ? kNoTile : (second ? -2 - t : t);
        bars->codes[it & 7] = code;
        if (code == kNoTile) {
          tc::mbar_arrive(&bars->full[s]);  // no copy: the consumers see the end
          break;
        }
        tc::mbar_arrive_expect_tx(&bars->full[s], (uint32_t)G::kTileBytes);
        for (int h = 0; h < G::KH; ++h)
          tc::tma_load_2d(ring + s * G::kTileBytes + h * kBoxBytes, &tk, h * 64,
                          krow + t * kTileKeys, &bars->full[s]);
        issued = it + 1;
        claim = info.nch + atomicAdd(ctr + (second ? 1 : 0), 1);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA
    // The whole warp runs the loop (barrier waits, descriptor arithmetic) and
    // one elected lane issues the MMAs and commits; the waits' outcome is made
    // warp-uniform so that every lane leaves the loop together.
    if (__all_sync(0xffffffffu, tc::mbar_wait(&bars->qfull, 0, abort, status))) {
      const uint32_t idesc2 = tc::idesc_bf16(128, NP);
      const uint64_t qdesc = tc::sw128_desc(tc::smem_addr(q_s));
      const uint64_t rdesc = tc::sw128_desc(tc::smem_addr(ring));
      for (int it = 0;; ++it) {
        const int s = it % kStages, a = it & 1;
        const bool ready = tc::mbar_wait(&bars->full[s], (it / kStages) & 1, abort, status) &&
                           tc::mbar_wait(&bars->tempty[a], ((it >> 1) & 1) ^ 1, abort, status);
        if (!__all_sync(0xffffffffu, ready)) break;
        tc::tc_fence_after();
        // the tile code travels with the accumulator to the epilogue
        const int code = reinterpret_cast<volatile int*>(bars->codes)[it & 7];
        if (lane == 0) reinterpret_cast<volatile int*>(bars->accode)[a] = code;
        __threadfence_block();
        const uint32_t on = tc::elect_one();
        if (code != kNoTile) {
          const uint64_t kdesc = desc_plus(rdesc, (uint32_t)(s * G::kTileBytes));
          const uint32_t dt = tmem + (uint32_t)(a * 256);
          mma_tile_steps<D, 0, G::kKSteps>(code >= 0, RB, dt, qdesc, kdesc, idesc2, on);
          tc::mma_commit_if(&bars->empty[s], on);
        }
        tc::mma_commit_if(&bars->tfull[a], on);
        committed = it + 1;
        if (code == kNoTile) break;
      }
    }
  } else if (warp < kEpiWarps) {
    // ---------------------------------------------------------------- epilogue
    const int sub = warp >> 2, quad = warp & 3;
    const float c = p.scale_log2;
    bool ok = true;
    int it = 0;  // accumulators consumed so far (both passes)

    if (MODE & kPassStats) {
      // rows: row block wg, TMEM lane quadrant quad; keys: half `half` of each tile
      const int wg = sub >> 1, half = sub & 1;
      const int row = wg * 128 + quad * 32 + lane;
      const int w = row % p.window;
      const int vis_end = min(rq.n, rq.p + w + 1);  // keys [0, vis_end) visible to the row
      float m_run = -INFINITY;
      float l_run = 0.f, l_comp = 0.f;  // compensated running sum of 2^(t - m_run)
      for (;; ++it) {
        const int a = it & 1;
        if (!tc::mbar_wait(&bars->tfull[a], (it >> 1) & 1, abort, status)) {
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const int code = reinterpret_cast<volatile int*>(bars->accode)[a];
        if (code < 0) break;  // a pass 2 tile or the end: pass 2 takes it from here
        const int t = code;
        bool released = false;
        if (wg < RB) {
          const uint32_t taddr =
              tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(a * 256 + wg * 128 + half * 64);
          const int key0 = t * kTileKeys + half * 64;
          const bool all_vis = (t + 1) * kTileKeys <= rq.p;
          // this warp's 64 columns of the tile: two TMEM loads, one wait
          float v[64];
          __syncwarp();
          tc::tmem_ld32(taddr, *reinterpret_cast<float(*)[32]>(v));
          tc::tmem_ld32(taddr + 32, *reinterpret_cast<float(*)[32]>(v + 32));
          tc::tmem_ld_wait();
          // the values are in registers: hand the accumulator back to the MMA
          // warp before computing, so the next-but-one tile's MMAs can start
          tc::tc_fence_before();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_rx(&bars->tempty[a]);
          released = true;
          if (!all_vis) {
#pragma unroll
            for (int i = 0; i < 64; ++i)
              if (key0 + i >= vis_end) v[i] = -INFINITY;
          }
          // slab max with three-input max
          float mt[22];
#pragma unroll
          for (int i = 0; i < 21; ++i) mt[i] = tc::max3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
          mt[21] = v[63];
          float mu[8];
#pragma unroll
          for (int i = 0; i < 7; ++i) mu[i] = tc::max3(mt[3 * i], mt[3 * i + 1], mt[3 * i + 2]);
          mu[7] = mt[21];
          const float mx = tc::max3(tc::max3(mu[0], mu[1], mu[2]), tc::max3(mu[3], mu[4], mu[5]),
                                    fmaxf(mu[6], mu[7]));
          const float m_new = fmaxf(m_run, mx * c);
          if (m_new != -INFINITY) {  // some key of this slab is visible
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
            for (int i = 0; i < 64; i += 4) {
              const float2 x = tc::upk2(tc::fma2(tc::pk2(v[i], v[i + 1]), cc, mm));
              const float2 y = tc::upk2(tc::fma2(tc::pk2(v[i + 2], v[i + 3]), cc, mm));
              acc0 = tc::add2(acc0, tc::pk2(fast_exp2(x.x), fast_exp2(x.y)));
              acc1 = tc::add2(acc1, tc::pk2(fast_exp2(y.x), fast_exp2(y.y)));
            }
            const float2 s01 = tc::upk2(tc::add2(acc0, acc1));
            const float term = (s01.x + s01.y) - l_comp;
            const float tsum = l_run + term;
            l_comp = (tsum - l_run) - term;
            l_run = tsum;
          }
        }
        if (!released) {
          tc::tc_fence_before();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_rx(&bars->tempty[a]);
        }
      }
      // the second column half hands its (max, sum) to the first
      if (half == 1) {
        if (ok) mrg[row] = make_float2(m_run, l_run);
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&bars->mrg);
      } else {
        ok = ok && tc::mbar_wait(&bars->mrg, 0, abort, status);
        if (ok && wg < RB && row < M) {
          const float2 o = mrg[row];
          const float m = fmaxf(m_run, o.x);
          const float l =
              (m == -INFINITY) ? 0.f : l_run * fast_exp2(m_run - m) + o.y * fast_exp2(o.x - m);
          partial[(size_t)item * M + row] = make_float2(m, l);
          if (kSums && l > 0.f) {
            // the row's sum over the whole grid, sum_c l_c 2^(m_c), in fp64 (no
            // common reference needed: 2^m stays finite for |m| < 960, which
            // leaves room for the sum); larger rows take the slow merge
            if (fabsf(m) < 960.f) {
              // l 2^m = (l 2^f) 2^i with m = i + f, f in [0, 1): the fp32
              // factors multiply exactly in fp64, the power of two is a scale
              const float fi = floorf(m);
              const double two_i = __longlong_as_double((long long)(1023 + (int)fi) << 52);
              atomicAdd(&lsum[segrow + row], (double)l * (double)exp2f(m - fi) * two_i);
            } else {
              atomicOr(gsync, kSumOverflowBit);  // read with the barrier count
            }
          }
        }
      }
    }

    if (kFused) {
      // publish this CTA's partials, then meet the grid (one thread waits).
      // The writers need no fence of their own: __syncwarp orders each lane's
      // writes before lane 0's arrive (a CTA-scope release), the waiter's
      // acquire then precedes its GPU-scope fence and arrival, and that
      // release is cumulative over everything ordered before it.
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->pub);
      if (warp == 0 && lane == 0) {
        if (tc::mbar_wait(&bars->pub, 0, abort, status) && !*abort) {
          __threadfence();
          atomicAdd(gsync, 1u);
          const uint64_t t0 = tc::globaltimer();
          uint32_t seen;
          while (((seen = ld_acquire(gsync)) & (kSums ? ~kSumOverflowBit : ~0u)) < gridDim.x) {
            if (*abort) break;
            if (tc::globaltimer() - t0 > tc::kWaitNs) {
              *abort = 1;
              atomicOr(status, kStatusTimeout);
              break;
            }
            __nanosleep(64);
          }
          if (kSums) bars->sums_ok = (seen & kSumOverflowBit) == 0;
        }
        tc::mbar_arrive(&bars->gready);  // also on abort: the waiters then see the flag
      }
      ok = ok && tc::mbar_wait(&bars->gready, 0, abort, status) && !*abort;
      // -c_row of every window row: log2 of its fp64 grid sum, or, when a row
      // maximum was out of that range, the merge of every chunk's partial
      if (kSums && ok && bars->sums_ok) {
        if (threadIdx.x < 256) {
          const int r = threadIdx.x;
          float v = -INFINITY;
          if (r < M) {
            // log2 of the fp64 sum: its binary exponent plus log2 of the
            // mantissa in [1, 2), the latter in fp32
            const long long bits = __double_as_longlong(__ldcg(&lsum[segrow + r]));
            const int e = (int)((bits >> 52) & 0x7ff) - 1023;
            const float mant = (float)__longlong_as_double((bits & 0x000fffffffffffffLL) |
                                                           0x3ff0000000000000LL);
            v = -((float)e + log2f(mant));
          }
          debug_flag(r < M && !isfinite(v), status);  // a row normaliser out of range
          ncr[r] = v;
        }
      } else if (ok) {
        const size_t it0 = (size_t)rq.item0 + (size_t)info.g * info.nch;
        // two threads per window row (adjacent lanes) fold alternate CTAs'
        // partials in one pass (online rescaling, compensated sums), then
        // combine through a shuffle in a fixed order
        const int r = threadIdx.x >> 1, part = threadIdx.x & 1;
        float m = -INFINITY, l = 0.f, comp = 0.f;
        if (r < M) {
#pragma unroll 4
          for (int ch = part; ch < info.nch; ch += 2) {
            const float2 pv = __ldcg(&partial[(it0 + ch) * M + r]);
            if (pv.y > 0.f) {
              if (pv.x > m) {
                const float sc = exp2f(m - pv.x);
                l *= sc;
                comp *= sc;
                m = pv.x;
              }
              const float term = pv.y * exp2f(pv.x - m) - comp;
              const float tsum = l + term;
              comp = (tsum - l) - term;
              l = tsum;
            }
          }
        }
        const float mo = __shfl_xor_sync(0xffffffffu, m, 1);
        const float lo = __shfl_xor_sync(0xffffffffu, l, 1);
        if (part == 0) {
          float v = -INFINITY;
          if (r < M) {
            const float mm = fmaxf(m, mo);
            const float ll = (l > 0.f ? l * exp2f(m - mm) : 0.f) + (lo > 0.f ? lo * exp2f(mo - mm) : 0.f);
            v = -(mm + log2f(ll));
          }
          debug_flag(r < M && !isfinite(v), status);  // a row normaliser out of range
          ncr[r] = v;
        }
      }
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&bars->crdone);
      ok = ok && tc::mbar_wait(&bars->crdone, 0, abort, status);
    }

    if ((MODE & kPassVotes) && ok) {
      // keys: TMEM lane quadrant quad; window rows (columns): quarter `sub`
      const int key = quad * 32 + lane;  // TMEM lane = key within the tile
      int pend_j = -1;  // a reduction not yet issued
      float pend_v = 0.f;
      for (;; ++it) {
        const int a = it & 1;
        if (!tc::mbar_wait(&bars->tfull[a], (it >> 1) & 1, abort, status)) break;
        tc::tc_fence_after();
        const int code = reinterpret_cast<volatile int*>(bars->accode)[a];
        if (code == kNoTile) break;  // the MMA warp has finished
        const int t = -2 - code;
        const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(a * 256);
        float acc = 0.f;
        bool released = false;
        const int c0 = sub * 64;
        if (c0 < NP) {
          // this warp's (up to) 64 window-row columns: two TMEM loads, one wait
          float v[64];
          __syncwarp();
          tc::tmem_ld32(taddr + c0, *reinterpret_cast<float(*)[32]>(v));
          if (c0 + 32 < NP) tc::tmem_ld32(taddr + c0 + 32, *reinterpret_cast<float(*)[32]>(v + 32));
          tc::tmem_ld_wait();
          // the previous tile's reduction, issued after this wait (a TMEM
          // load wait issued behind a global store waits for it)
          if (pend_j >= 0) {
            atomicAdd(sc_out + pend_j, pend_v);
            pend_j = -1;
          }
          tc::tc_fence_before();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_rx(&bars->tempty[a]);
          released = true;
          // 2^(v c - c_row) over the columns the MMA wrote: NP - c0 is a
          // multiple of 16, and columns past NP were never written
          const int nv = min(64, NP - c0);
          acc = nv == 64   ? vote_sum<64>(v, c, ncr + c0)
                : nv == 48 ? vote_sum<48>(v, c, ncr + c0)
                : nv == 32 ? vote_sum<32>(v, c, ncr + c0)
                           : vote_sum<16>(v, c, ncr + c0);
        }
        if (!released) {
          tc::tc_fence_before();
          __syncwarp();
          if (lane == 0) tc::mbar_arrive_rx(&bars->tempty[a]);
        }
        // this warp's quarter of the window rows, added into the key's score
        const int j = t * kTileKeys + key;
        if (sub * 64 < NP && j < rq.p) {
          pend_j = j;
          pend_v = acc;
        }
      }
      if (pend_j >= 0) atomicAdd(sc_out + pend_j, pend_v);
    }
  }

  // ---- teardown: drain what is still in flight, release TMEM
  if (warp == kProducerWarp && lane == 0 && *abort) {
    int dummy = 0;
    tc::mbar_wait(&bars->qfull, 0, &dummy, status);
    for (int s = 0; s < kStages && s < issued; ++s) {
      const int last = issued - 1 - ((issued - 1 - s) % kStages);
      tc::mbar_wait(&bars->full[s], (uint32_t)((last / kStages) & 1), &dummy, status);
    }
  }
  if (warp == kMmaWarp && lane == 0 && committed > 0) {
    // the last accumulator commit covers every MMA this thread issued
    const int last = committed - 1;
    int dummy = 0;
    tc::mbar_wait(&bars->tfull[last & 1], (uint32_t)((last >> 1) & 1), &dummy, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == kProducerWarp) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
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

// CTAs of the fused kernel that fit on the current device at once (cached).
int coresident_ctas(const void* kernel, int smem, int slot) {
  constexpr int kMaxDev = 64;
  static int cache[kMaxDev][2] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev][slot] == 0) {
    int sms = 0, per_sm = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, smem) !=
            cudaSuccess)
      return 0;
    cache[dev][slot] = sms * per_sm;
  }
  return cache[dev][slot];
}

template <int D>
cudaError_t launch_tc_typed(const EvictParams& pt, const CUtensorMap& tq, const CUtensorMap& tk,
                            float* scores, float2* partial, float* rowc, int32_t* status,
                            int32_t* tilectr, double* lsum, cudaStream_t s) {
  using Gm = Geo<D>;
  uint32_t* gsync = reinterpret_cast<uint32_t*>(status) + kGridSyncWord;
  constexpr int kRv = kRedVotes;
  auto fused = window_scores_row_sums(pt) ? ws_tc<D, kPassBoth | kRowSums | kRv>
                                          : ws_tc<D, kPassBoth | kRv>;
  cudaError_t e =
      cudaFuncSetAttribute(fused, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  if (pt.items <= coresident_ctas(reinterpret_cast<const void*>(fused), Gm::kSmem, D == 128)) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)pt.items, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = Gm::kSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, fused, pt, tq, tk, partial, (const float*)rowc, scores, status,
                           gsync, tilectr, lsum);
    count_launches(1);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  // fallback: the passes as separate launches with the merge kernel between
  auto stats = ws_tc<D, kPassStats | kRv>;
  auto votes = ws_tc<D, kPassVotes | kRv>;
  e = cudaFuncSetAttribute(stats, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(votes, cudaFuncAttributeMaxDynamicSharedMemorySize, Gm::kSmem);
  if (e != cudaSuccess) return e;
  stats<<<pt.items, kThreads, Gm::kSmem, s>>>(pt, tq, tk, partial, rowc, scores, status, gsync,
                                              tilectr, (double*)nullptr);
  e = launch_window_combine(pt, partial, rowc, s);
  if (e != cudaSuccess) return e;
  votes<<<pt.items, kThreads, Gm::kSmem, s>>>(pt, tq, tk, partial, rowc, scores, status, gsync,
                                              tilectr, (double*)nullptr);
  count_launches(2);
  return cudaGetLastError();
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
  for (int b = 0; b < p.batch; ++b)
    tiles += (int64_t)p.hkv * ((p.req[b].n + kTileKeys - 1) / kTileKeys);
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
                                    int32_t* tilectr, double* lsum, cudaStream_t s) {
  const EvictParams pt = tc_item_params(p);
  CUtensorMap tq, tk;
  const uint64_t qrows = (uint64_t)p.batch * p.hq * p.window;
  const uint64_t krows = (uint64_t)p.hkv * p.kv_rows;
  if (!make_bf16_map(&tq, q_win, p.d, qrows, 128) || !make_bf16_map(&tk, K, p.d, krows, 128))
    return cudaErrorInvalidValue;
  return p.d == 64
             ? launch_tc_typed<64>(pt, tq, tk, scores, partial, rowc, status, tilectr, lsum, s)
             : launch_tc_typed<128>(pt, tq, tk, scores, partial, rowc, status, tilectr, lsum, s);
}

cudaError_t launch_window_votes_tc(const EvictParams& p, const void* q_win, const void* K,
                                   float* scores, const float* rowc, int32_t* status,
                                   int32_t* tilectr, cudaStream_t s) {
  const EvictParams pt = tc_item_params(p);
  CUtensorMap tq, tk;
  const uint64_t qrows = (uint64_t)p.batch * p.hq * p.window;
  const uint64_t krows = (uint64_t)p.hkv * p.kv_rows;
  if (!make_bf16_map(&tq, q_win, p.d, qrows, 128) || !make_bf16_map(&tk, K, p.d, krows, 128))
    return cudaErrorInvalidValue;
  uint32_t* gsync = reinterpret_cast<uint32_t*>(status) + kGridSyncWord;
  auto launch = [&](auto kern, int smem) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(kern, dim3(pt.items), dim3(kThreads), smem, s, pt, tq, tk, (float2*)nullptr, rowc,
                   scores, status, gsync, tilectr, (double*)nullptr);
    count_launches(1);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  };
  // the caller cleared the scores (with the workspace's control words)
  return p.d == 64 ? launch(ws_tc<64, kPassVotes | kRedVotes>, Geo<64>::kSmem)
                   : launch(ws_tc<128, kPassVotes | kRedVotes>, Geo<128>::kSmem);
}

bool window_scores_row_sums(const EvictParams& p) {
  if (!window_scores_tc_supported(p)) return false;
  const EvictParams pt = tc_item_params(p);
  for (int b = 0; b < p.batch; ++b)
    if ((p.req[b].n + pt.chunk - 1) / pt.chunk > kSumMinChunks) return true;
  return false;
}

}  // namespace tb
