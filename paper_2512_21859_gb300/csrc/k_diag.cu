// Diagnostic of the bounded device-side waits (failure detection).
//
// Every kernel of the library waits on mbarriers through tc::mbar_wait, which
// gives up after a time limit, raises the CTA's abort flag and the workspace
// status word, and lets the kernel drain its own copies, free its tensor
// memory and return. A real kernel only times out when something is broken,
// so this one reproduces the pattern on purpose, with nothing broken on the
// GPU: one CTA allocates tensor memory, starts one bulk copy into shared
// memory, then waits on an mbarrier that nothing arrives on (unless asked
// to arrive itself) with the caller's short limit; on timeout it takes the
// same exit as the real kernels (flag, drain, dealloc, return).
#include <cuda_runtime.h>

#include "tb_internal.cuh"
#include "tc_ptx.cuh"

namespace tb {
namespace {

constexpr uint32_t kDiagCopyBytes = 4096;
constexpr uint32_t kDiagTmemCols = 32;

__global__ void __launch_bounds__(64, 1)
    wait_diag(const uint8_t* __restrict__ src, int32_t* __restrict__ status, uint64_t limit_ns,
              int32_t arrive) {
  __shared__ __align__(16) uint8_t buf[kDiagCopyBytes];
  __shared__ uint64_t copy_bar, never_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  const int warp = threadIdx.x / 32;
  if (threadIdx.x == 0) {
    tc::mbar_init(&copy_bar, 1);
    tc::mbar_init(&never_bar, 1);
    abort_flag = 0;
    tc::fence_barrier_init();
  }
  if (warp == 0) tc::tmem_alloc(&tmem_base, kDiagTmemCols);
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  if (threadIdx.x == 0) {
    tc::mbar_arrive_expect_tx(&copy_bar, kDiagCopyBytes);
    tc::bulk_load(buf, src, kDiagCopyBytes, &copy_bar);
    if (arrive) tc::mbar_arrive(&never_bar);
    // the wait under test: returns false after limit_ns unless the arrive
    // above completed the phase
    tc::mbar_wait(&never_bar, 0, &abort_flag, status, limit_ns);
    // the exit every kernel takes: wait (bounded, with the library's own
    // limit) for this CTA's own copy before the CTA may end
    int dummy = 0;
    tc::mbar_wait(&copy_bar, 0, &dummy, status);
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem_base, kDiagTmemCols);
  }
}

}  // namespace
}  // namespace tb

using namespace tb;

extern "C" tb_status tb_diag_bounded_wait(void* workspace, size_t workspace_bytes,
                                          uint64_t limit_ns, int32_t arrive,
                                          tb_stream_t stream) {
  if (!workspace || workspace_bytes < kStatusBytes + kDiagCopyBytes ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return TB_ERR_WORKSPACE;
  if (limit_ns < 10000ull || limit_ns > 1000000000ull || (arrive != 0 && arrive != 1))
    return TB_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  tb_status st = cuda_status(clear_control_words(workspace, kStatusBytes, s));
  if (st != TB_OK) return st;
  const uint8_t* src = static_cast<const uint8_t*>(workspace) + kStatusBytes;
  wait_diag<<<1, 64, 0, s>>>(src, static_cast<int32_t*>(workspace), limit_ns, arrive);
  count_launches(1);
  return cuda_status(cudaGetLastError());
}
