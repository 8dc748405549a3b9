// Gather / compaction of the retained K and V rows.
//
//   Kc[g][out_off_b + r] = K[g][kv_off_b + idx[g][idx_off_b + r]],  r < R_b,
// and the same for V: pure bit copies in 16-byte vectors. One warp moves one
// retained row of K and the matching row of V; a row is d * elem bytes
// (128..512 B), so each 16-byte lane access is part of a fully used sector.
#include <cuda_runtime.h>

#include "tb_internal.cuh"

namespace tb {
namespace {

constexpr int kGatherThreads = 256;
constexpr int kRowsPerWarp = 4;

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(
    const __grid_constant__ EvictParams p, const int32_t* __restrict__ idx,
    const uint4* __restrict__ K, const uint4* __restrict__ V, uint4* __restrict__ Kc,
    uint4* __restrict__ Vc, int vec_per_row) {
  const int b = blockIdx.y, g = blockIdx.z;
  const EvictReq& rq = p.req[b];
  const int R = rq.k + p.window;
  const int lane = threadIdx.x & 31;
  const int warp_global = (blockIdx.x * kGatherThreads + threadIdx.x) >> 5;
  const int32_t* ig = idx + (size_t)g * p.idx_rows + rq.idx_off;
  const size_t src_base = ((size_t)g * p.kv_rows + rq.kv_off) * vec_per_row;
  const size_t dst_base = ((size_t)g * p.out_rows + rq.out_off) * vec_per_row;
  for (int rr = 0; rr < kRowsPerWarp; ++rr) {
    const int r = warp_global * kRowsPerWarp + rr;
    if (r >= R) return;
    const int j = __ldg(ig + r);
    if (j < 0 || j >= rq.n) continue;
    const uint4* ks = K + src_base + (size_t)j * vec_per_row;
    const uint4* vs = V + src_base + (size_t)j * vec_per_row;
    uint4* kd = Kc + dst_base + (size_t)r * vec_per_row;
    uint4* vd = Vc + dst_base + (size_t)r * vec_per_row;
    for (int v = lane; v < 2 * vec_per_row; v += 32) {
      if (v < vec_per_row) {
        kd[v] = __ldg(ks + v);
      } else {
        vd[v - vec_per_row] = __ldg(vs + v - vec_per_row);
      }
    }
  }
}

}  // namespace

cudaError_t launch_gather(const EvictParams& p, const int32_t* idx, const void* K,
                          const void* V, void* Kc, void* Vc, cudaStream_t s) {
  const int elem = p.dtype == TB_F32 ? 4 : 2;
  const int vec_per_row = p.d * elem / 16;
  const int rows_per_block = (kGatherThreads / 32) * kRowsPerWarp;
  const int bx = (p.max_r + rows_per_block - 1) / rows_per_block;
  if (bx == 0) return cudaSuccess;
  dim3 grid(bx, p.batch, p.hkv);
  gather_kernel<<<grid, kGatherThreads, 0, s>>>(
      p, idx, static_cast<const uint4*>(K), static_cast<const uint4*>(V),
      static_cast<uint4*>(Kc), static_cast<uint4*>(Vc), vec_per_row);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace tb
