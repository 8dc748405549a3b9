// Gather / compaction of the retained K and V rows.
//
//   Kc[g][out_off_b + r] = K[g][kv_off_b + idx[g][idx_off_b + r]],  r < R_b,
// and the same for V: pure bit copies in 16-byte vectors. A row is d * elem
// bytes (128..512 B), so each 16-byte lane access is part of a fully used
// sector.
#include <cuda_runtime.h>

#include "tb_internal.cuh"

namespace tb {
namespace {

constexpr int kGatherThreads = 256;
// Four rows per warp: measured on GB300 against eight, the gather alone took
// 128K 20.6 -> 19.6 us and 32K 13.1 -> 12.4 us, and beside a select and a
// decode (fewer registers per block, so more blocks fit beside them) the
// pipelined step 142.3 -> 140.5 us and 49.7 -> 47.1 us; two rows per warp, or
// 512-thread blocks, were no better.
constexpr int kRowsPerWarp = 4;
constexpr int kMaxVecPerLane = 16;  // kRowsPerWarp * 2 rows * up to 32 vectors / 32 lanes

// Each warp moves kRowsPerWarp retained rows of K and the matching rows of V:
// first every lane issues all of its 16-byte loads, then all of its stores,
// so that each lane keeps several independent loads in flight.
template <int VPR>
__device__ __forceinline__ void gather_rows(const EvictParams& p, const int32_t* __restrict__ idx,
                                            const uint4* __restrict__ K, const uint4* __restrict__ V,
                                            uint4* __restrict__ Kc, uint4* __restrict__ Vc,
                                            int32_t* __restrict__ status) {
  constexpr int kVecs = kRowsPerWarp * 2 * VPR;  // vectors a warp moves
  constexpr int kPerLane = kVecs / 32;
  static_assert(kPerLane <= kMaxVecPerLane, "too many vectors per lane");
  const int b = blockIdx.y, g = blockIdx.z;
  const EvictReq& rq = p.req[b];
  const int R = rq.k + p.window;
  const int lane = threadIdx.x & 31;
  const int r0 = ((blockIdx.x * kGatherThreads + threadIdx.x) >> 5) * kRowsPerWarp;
  if (r0 >= R) return;
  const int32_t* ig = idx + (size_t)g * p.idx_rows + rq.idx_off;
  const size_t src_base = ((size_t)g * p.kv_rows + rq.kv_off) * VPR;
  const size_t dst_base = ((size_t)g * p.out_rows + rq.out_off) * VPR;
  uint4 buf[kPerLane];
  bool ok[kPerLane];
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    const int v = lane + 32 * i;
    const int rr = v / (2 * VPR), w = v % (2 * VPR);
    const int r = r0 + rr;
    int j = -1;
    if (r < R) j = __ldg(ig + r);
    ok[i] = r < R && j >= 0 && j < rq.n;
    debug_flag(r < R && !ok[i], status);  // an index outside the request's rows
    if (ok[i]) {
      const uint4* src = (w < VPR ? K : V) + src_base + (size_t)j * VPR + (w < VPR ? w : w - VPR);
      buf[i] = __ldg(src);
    }
  }
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    if (!ok[i]) continue;
    const int v = lane + 32 * i;
    const int rr = v / (2 * VPR), w = v % (2 * VPR);
    uint4* dst = (w < VPR ? Kc : Vc) + dst_base + (size_t)(r0 + rr) * VPR + (w < VPR ? w : w - VPR);
    *dst = buf[i];
  }
}

template <int VPR>
__global__ void __launch_bounds__(kGatherThreads) gather_kernel(
    const __grid_constant__ EvictParams p, const int32_t* __restrict__ idx,
    const uint4* __restrict__ K, const uint4* __restrict__ V, uint4* __restrict__ Kc,
    uint4* __restrict__ Vc, int32_t* __restrict__ status) {
  // idx comes from the select kernel just before, unless the caller asserts
  // (TB_EVICT_GATHER_CONCURRENT) that the kernel before writes none of it
  const bool concurrent = p.flags & TB_EVICT_GATHER_CONCURRENT;
  if (!concurrent) pdl_wait();
  pdl_trigger();
  gather_rows<VPR>(p, idx, K, V, Kc, Vc, status);
  // A concurrent gather waits for the kernel before it only now, in one
  // thread after all of its block's copies, so that the grid still completes
  // after that kernel: whatever waits for the gather waits for both. That
  // kernel's CTAs have all started (it let this grid launch only then), so
  // the wait ends.
  if (concurrent && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 && threadIdx.x == 0)
    pdl_wait();
}

}  // namespace

cudaError_t launch_gather(const EvictParams& p, const int32_t* idx, const void* K,
                          const void* V, void* Kc, void* Vc, int32_t* status, cudaStream_t s) {
  const int elem = p.dtype == TB_F32 ? 4 : 2;
  const int vec_per_row = p.d * elem / 16;
  const int rows_per_block = (kGatherThreads / 32) * kRowsPerWarp;
  const int bx = (p.max_r + rows_per_block - 1) / rows_per_block;
  if (bx == 0) return cudaSuccess;
  dim3 grid(bx, p.batch, p.hkv);
  const uint4* k4 = static_cast<const uint4*>(K);
  const uint4* v4 = static_cast<const uint4*>(V);
  uint4* kc4 = static_cast<uint4*>(Kc);
  uint4* vc4 = static_cast<uint4*>(Vc);
  cudaError_t e;
  switch (vec_per_row) {
    case 8: e = launch_pdl(gather_kernel<8>, grid, dim3(kGatherThreads), 0, s, p, idx, k4, v4, kc4, vc4, status); break;
    case 16: e = launch_pdl(gather_kernel<16>, grid, dim3(kGatherThreads), 0, s, p, idx, k4, v4, kc4, vc4, status); break;
    case 32: e = launch_pdl(gather_kernel<32>, grid, dim3(kGatherThreads), 0, s, p, idx, k4, v4, kc4, vc4, status); break;
    default: return cudaErrorInvalidValue;
  }
  count_launches(1);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace tb
