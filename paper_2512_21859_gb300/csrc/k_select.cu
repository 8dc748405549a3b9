// Max-pool and per-head top-k selection with ordered compaction.
//
// Pool[j] = max of S over [j - pool_k/2, j + pool_k/2] clipped to the prefix
// (stride 1, out-of-range neighbours ignored), or with TB_EVICT_AVG_POOL the
// sum over that range / pool_k (out-of-range neighbours count as zeros; the
// selection ranks the sums, whose order is the averages' order, and only the
// pooled output is scaled). Then, per (request, KV head),
// the k largest pooled scores are kept, ties to the lower index, and written
// in ascending index order followed by the window positions P..N-1.
//
// Selection is a most-significant-digit radix select on the float bit
// pattern (scores are >= 0, so unsigned order equals numeric order): four
// 8-bit digit histograms find the k-th largest value tau and how many of the
// tau-valued entries to keep; one ordered pass then keeps every entry above
// tau and the first `need` entries equal to tau, which yields sorted indices
// without a sort.
#include <cooperative_groups.h>
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
  const bool avg = (p.flags & TB_EVICT_AVG_POOL) != 0;
  const float inv = 1.0f / (float)p.pool_k;
  const size_t base = (size_t)g * p.score_rows + rq.score_off;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < P; j += gridDim.x * blockDim.x) {
    const int lo = max(0, j - half), hi = min(P - 1, j + half);
    float m = scores[base + lo];
    for (int t = lo + 1; t <= hi; ++t) m = avg ? m + scores[base + t] : fmaxf(m, scores[base + t]);
    pooled[base + j] = avg ? m * inv : m;
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
                                                             int32_t* __restrict__ idx,
                                                             int32_t* __restrict__ status) {
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
    debug_flag(sel && pos >= k, status);
    base_sel += tot_sel;
    base_tie += tot_eq;
  }
  debug_flag(tid == 0 && base_sel != k, status);  // exactly k positions kept
}


// ---------------------------------------------------------------------------
// Cluster select: one thread-block cluster of `cs` CTAs per (request, KV head)
// segment. CTA r of the cluster owns prefix positions [r*L, r*L + L): it loads
// that slice of the scores with a pool_k/2 halo into shared memory, max-pools
// it in place, and keeps the pooled bit patterns there. The four radix passes
// build a 256-bin histogram per CTA; every CTA sums the cluster's histograms
// through distributed shared memory and derives the same digit. Compaction
// runs warp by warp over contiguous runs with ballots, after one exchange of
// per-CTA (greater, equal) counts fixes each CTA's output offset.
// ---------------------------------------------------------------------------
constexpr int kCsThreads = 1024;
constexpr int kCsWarps = kCsThreads / 32;

// 32-key chunks of one warp's run in the compaction (runs of up to 512 keys)
constexpr int kRunChunks = kClusterSliceMax / kCsThreads;

struct ClusterSelectShared {
  unsigned hist[2][256];
  uint2 masks[kCsWarps][kRunChunks];  // per chunk: ballots of (key > tau, key == tau)
  unsigned total[256];
  int wgt[kCsWarps], weq[kCsWarps];
  int cta_cnt[2];  // this CTA's (greater, equal) counts, read by the cluster
  int rank_cnt[8][2];  // the lower ranks' counts (cluster size <= 8)
  unsigned prefix;
  int need;
};

__global__ void __launch_bounds__(kCsThreads) select_cluster_kernel(
    const __grid_constant__ EvictParams p, const float* __restrict__ scores,
    float* __restrict__ pooled_out, int32_t* __restrict__ idx, int32_t* __restrict__ status,
    int slice) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  __shared__ ClusterSelectShared sh;
  extern __shared__ __align__(16) float keys_f[];  // slice + 2 * halo floats (+ slack)
  unsigned* keys = reinterpret_cast<unsigned*>(keys_f);

  const int cs = (int)cluster.num_blocks();
  const int rank = (int)cluster.block_rank();
  const int seg = blockIdx.x / cs;
  const int b = seg / p.hkv, g = seg % p.hkv;
  const EvictReq& rq = p.req[b];
  const int P = rq.p, k = rq.k, half = p.pool_k / 2;
  const bool avg = (p.flags & TB_EVICT_AVG_POOL) != 0;
  const int lo = min(P, rank * slice);
  const int cnt = max(0, min(P, lo + slice) - lo);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();  // the scores come from the kernel just before
  pdl_trigger();
  const float* S = scores + (size_t)g * p.score_rows + rq.score_off;
  int32_t* out = idx + (size_t)g * p.idx_rows + rq.idx_off;

  if (rank == 0)
    for (int t = tid; t < p.window; t += kCsThreads) out[k + t] = P + t;

  // slice + halo, -inf outside the prefix for max-pooling (scores are >= 0,
  // so max is exact), 0 for average pooling; four loads in flight per thread
  const float pad = avg ? 0.f : -INFINITY;
  const int nin = cnt + 2 * half;
  for (int i0 = tid; i0 < nin; i0 += 4 * kCsThreads) {
    float x[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * kCsThreads, j = lo - half + i;
      x[q] = (i < nin && j >= 0 && j < P) ? S[j] : pad;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + q * kCsThreads;
      if (i < nin) keys_f[i] = x[q];
    }
  }
  __syncthreads();
  constexpr int kMaxPer = kClusterSliceMax / kCsThreads;
  unsigned reg[kMaxPer];
  // pool_k = 7, max: each thread pools groups of four consecutive outputs
  // 4q .. 4q+3 from the ten inputs keys_f[4q .. 4q+9], read as three 16-byte
  // vectors (the smem array has slack past its inputs for the last group's
  // vectors; values there only reach outputs >= cnt, which are not kept).
  // Three vector loads per four outputs instead of seven scalar loads per
  // output: the pooling is bound by shared-memory wavefronts.
  const bool grouped = half == 3 && !avg;
  if (grouped) {
#pragma unroll
    for (int r = 0; r < kMaxPer / 4; ++r) {
      const int q = tid + r * kCsThreads;
      if (4 * q < cnt) {
        const float4 u = *reinterpret_cast<const float4*>(keys_f + 4 * q);
        const float4 v = *reinterpret_cast<const float4*>(keys_f + 4 * q + 4);
        const float4 w = *reinterpret_cast<const float4*>(keys_f + 4 * q + 8);
        // inputs x0..x9 = u.x u.y u.z u.w v.x v.y v.z v.w w.x w.y; output k is
        // the max of x_k .. x_{k+6}, all four share x3..x6
        const float core = fmaxf(fmaxf(u.w, v.x), fmaxf(v.y, v.z));
        const float m12 = fmaxf(u.y, u.z), m78 = fmaxf(v.w, w.x);
        reg[4 * r + 0] = __float_as_uint(fmaxf(fmaxf(core, u.x), m12));
        reg[4 * r + 1] = __float_as_uint(fmaxf(fmaxf(core, m12), v.w));
        reg[4 * r + 2] = __float_as_uint(fmaxf(fmaxf(core, u.z), m78));
        reg[4 * r + 3] = __float_as_uint(fmaxf(fmaxf(core, m78), w.y));
      }
    }
  } else if (half == 3) {  // the same window, summed in a fixed order
#pragma unroll
    for (int r = 0; r < kMaxPer; ++r) {
      const int i = tid + r * kCsThreads;
      if (i < cnt) {
        const float* x = keys_f + i;
        reg[r] = __float_as_uint(((x[0] + x[1]) + (x[2] + x[3])) + ((x[4] + x[5]) + x[6]));
      }
    }
  } else {
#pragma unroll
    for (int r = 0; r < kMaxPer; ++r) {
      const int i = tid + r * kCsThreads;
      if (i < cnt) {
        float m = keys_f[i];
        for (int t = 1; t <= 2 * half; ++t) m = avg ? m + keys_f[i + t] : fmaxf(m, keys_f[i + t]);
        reg[r] = __float_as_uint(m);
      }
    }
  }
  __syncthreads();
  if (grouped) {
#pragma unroll
    for (int r = 0; r < kMaxPer / 4; ++r) {
      const int q = tid + r * kCsThreads;
      if (4 * q + 3 < cnt) {
        *reinterpret_cast<uint4*>(keys + 4 * q) =
            make_uint4(reg[4 * r], reg[4 * r + 1], reg[4 * r + 2], reg[4 * r + 3]);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (4 * q + k < cnt) keys[4 * q + k] = reg[4 * r + k];
      }
    }
  } else {
#pragma unroll
    for (int r = 0; r < kMaxPer; ++r) {
      const int i = tid + r * kCsThreads;
      if (i < cnt) keys[i] = reg[r];
    }
  }
  __syncthreads();
  if (pooled_out) {
    float* po = pooled_out + (size_t)g * p.score_rows + rq.score_off + lo;
    const float scale = avg ? 1.0f / (float)p.pool_k : 1.0f;
    for (int i = tid; i < cnt; i += kCsThreads) po[i] = __uint_as_float(keys[i]) * scale;
  }

  // every prefix position kept (alpha = 0, or a budget above the prefix):
  // the indices are the positions themselves, no selection or exchange
  if (k >= P) {
    for (int i = tid; i < cnt; i += kCsThreads) out[lo + i] = lo + i;
    return;
  }

  // ---- radix select of the k-th largest key (uniform across the cluster)
  unsigned tau = 0;
  int need = 0;
  const bool partial_sel = k > 0 && k < P;
  if (partial_sel) {
    unsigned prefix = 0, mask = 0;
    need = k;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      unsigned* h = sh.hist[pass & 1];
      for (int t = tid; t < 256; t += kCsThreads) h[t] = 0;
      __syncthreads();
      // four keys per round: their loads and digits are independent (the
      // kernel is bound by the latency of these loops, not by throughput)
      for (int i0 = tid; i0 < cnt; i0 += 4 * kCsThreads) {
        unsigned kv[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int i = i0 + q * kCsThreads;
          kv[q] = i < cnt ? keys[i] : 0u;
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int i = i0 + q * kCsThreads;
          if (i < cnt && (kv[q] & mask) == prefix) atomicAdd(&h[(kv[q] >> shift) & 255u], 1u);
        }
      }
      cluster.sync();
      if (tid < 256) {
        unsigned v[8];
#pragma unroll
        for (int r = 0; r < 8; ++r) v[r] = r < cs ? cluster.map_shared_rank(h, r)[tid] : 0u;
        sh.total[tid] = ((v[0] + v[1]) + (v[2] + v[3])) + ((v[4] + v[5]) + (v[6] + v[7]));
      }
      __syncthreads();
      if (warp == 0) {
        unsigned cntd[8], mine = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          cntd[i] = sh.total[255 - (lane * 8 + i)];
          mine += cntd[i];
        }
        unsigned inc = mine;
        for (int off = 1; off < 32; off <<= 1) {
          const unsigned o = __shfl_up_sync(0xffffffffu, inc, off);
          if (lane >= off) inc += o;
        }
        const unsigned above = inc - mine;
        if (above < (unsigned)need && inc >= (unsigned)need) {
          unsigned run = above;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            if (run + cntd[i] >= (unsigned)need) {
              sh.prefix = prefix | ((255u - (unsigned)(lane * 8 + i)) << shift);
              sh.need = need - (int)run;
              break;
            }
            run += cntd[i];
          }
        }
      }
      __syncthreads();
      prefix = sh.prefix;
      need = sh.need;
      mask |= 255u << shift;
    }
    tau = prefix;
  }

  // ---- ordered compaction over warp-contiguous runs
  const int run = ((cnt + kCsWarps - 1) / kCsWarps + 31) & ~31;
  const int wlo = min(cnt, warp * run), whi = min(cnt, wlo + run);
  int gt_w = 0, eq_w = 0;
  if (k > 0) {
    for (int b0 = wlo; b0 < whi; b0 += 128) {
      unsigned kv[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int i = b0 + 32 * q + lane;
        kv[q] = i < whi ? keys[i] : 0u;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int i = b0 + 32 * q + lane;
        const unsigned gm = __ballot_sync(0xffffffffu, i < whi && kv[q] > tau);
        const unsigned em = __ballot_sync(0xffffffffu, i < whi && kv[q] == tau);
        // the chunk's ballots, for the emission pass
        if (lane == q && b0 + 32 * q < whi) sh.masks[warp][(b0 - wlo) / 32 + q] = make_uint2(gm, em);
        gt_w += __popc(gm);
        eq_w += __popc(em);
      }
    }
  }
  if (lane == 0) {
    sh.wgt[warp] = gt_w;
    sh.weq[warp] = eq_w;
  }
  __syncthreads();
  if (warp == 0) {
    int gsum = sh.wgt[lane], esum = sh.weq[lane];
    for (int off = 16; off > 0; off >>= 1) {
      gsum += __shfl_xor_sync(0xffffffffu, gsum, off);
      esum += __shfl_xor_sync(0xffffffffu, esum, off);
    }
    if (lane == 0) {
      sh.cta_cnt[0] = gsum;
      sh.cta_cnt[1] = esum;
    }
  }
  cluster.sync();
  // the lower ranks' counts, all remote loads at once
  if (tid < 16) {
    const int r = tid >> 1;
    sh.rank_cnt[r][tid & 1] = r < rank ? cluster.map_shared_rank(sh.cta_cnt, r)[tid & 1] : 0;
  }
  __syncthreads();
  // no shared memory of another CTA is read after this point: arrive now, and
  // wait (so that none leaves while another may still read it) at the end
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  // offsets of this warp: ties are kept in index order until `need` are in,
  // so of the E ties before a point min(need, E) are kept, and the offsets
  // are prefix sums of the lower ranks' and warps' counts (one reduction
  // each, no chain through the warps)
  const int lg = (lane < rank ? sh.rank_cnt[lane & 7][0] : 0) + (lane < warp ? sh.wgt[lane] : 0);
  const int le = (lane < rank ? sh.rank_cnt[lane & 7][1] : 0) + (lane < warp ? sh.weq[lane] : 0);
  int eqbase = __reduce_add_sync(0xffffffffu, le);
  int selbase = __reduce_add_sync(0xffffffffu, lg) + min(need, eqbase);
  if (k > 0) {
    // emission from the count pass's ballots: per 32-key chunk, the keys
    // above tau and the first ties until `need` of them are kept
    const unsigned lt = (1u << lane) - 1u;
    const int nch = (whi - wlo + 31) / 32;
    for (int c = 0; c < nch; ++c) {
      const uint2 m = sh.masks[warp][c];
      const int room = need - eqbase;  // ties still to keep
      unsigned tie = room > 0 ? m.y : 0u;
      if (room > 0 && __popc(tie) > room)  // the chunk where the ties run out
        tie = __ballot_sync(0xffffffffu, ((m.y >> lane) & 1u) && __popc(m.y & lt) < room);
      const unsigned sm = m.x | tie;
      const int pos = selbase + __popc(sm & lt);
      const bool sel = (sm >> lane) & 1u;
      if (sel && pos < k) out[pos] = lo + wlo + 32 * c + lane;
      debug_flag(sel && pos >= k, status);
      selbase += __popc(sm);
      eqbase += __popc(m.y);
    }
  }
  // the cluster's last warp ends on the total: exactly k positions kept
  debug_flag(k > 0 && rank == cs - 1 && warp == kCsWarps - 1 && lane == 0 && selbase != k,
             status);
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
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
                          int32_t* status, cudaStream_t s) {
  select_kernel<<<p.batch * p.hkv, kSelThreads, 0, s>>>(p, pooled, idx, status);
  count_launches(1);
  return cudaGetLastError();
}

bool select_cluster_supported(const EvictParams& p) {
  const int cs = select_cluster_size(p);
  const int slice = (p.max_p + cs - 1) / cs;
  return slice <= kClusterSliceMax;
}

// One CTA per 4096 keys of the longest prefix, up to 8 (the portable cluster
// size): the kernel is bound by the latency of its phases, and on GB300 the
// smaller slices measured faster (32K keys: 23.6 -> 20.8 us with 8 CTAs).
int select_cluster_size(const EvictParams& p) {
  int cs = (p.max_p + 4095) / 4096;
  return cs < 1 ? 1 : (cs > 8 ? 8 : cs);
}

cudaError_t launch_select_cluster(const EvictParams& p, const float* scores, float* pooled_out,
                                  int32_t* idx, int32_t* status, cudaStream_t s) {
  const int cs = select_cluster_size(p);
  const int slice = (p.max_p + cs - 1) / cs;
  // slice + halo, plus slack for the grouped max-pool's last 16-byte loads
  const size_t smem = sizeof(float) * (((size_t)slice + 2 * (p.pool_k / 2) + 8 + 3) & ~(size_t)3);
  cudaError_t e = cudaFuncSetAttribute(select_cluster_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(p.batch * p.hkv * cs), 1, 1);
  cfg.blockDim = dim3(kCsThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  e = cudaLaunchKernelEx(&cfg, select_cluster_kernel, p, scores, pooled_out, idx, status, slice);
  count_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace tb
