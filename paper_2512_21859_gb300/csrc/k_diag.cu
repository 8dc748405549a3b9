// Diagnostic entry point: evaluates the FMA-pipe exponential the scoring
// epilogues use (tc::exp2_poly2) on a device array, so that tests can hold it
// against exact 2^x and against the MUFU exponential.
#include <cuda_runtime.h>

#include "tb_internal.cuh"
#include "tc_ptx.cuh"

namespace tb {
namespace {

__global__ void exp2_poly_kernel(const float* __restrict__ x, float* __restrict__ y, int64_t n) {
  const int64_t i = 2 * ((int64_t)blockIdx.x * blockDim.x + threadIdx.x);
  if (i + 1 < n) {
    const float2 r = tc::exp2_poly2(x[i], x[i + 1]);
    y[i] = r.x;
    y[i + 1] = r.y;
  } else if (i < n) {
    y[i] = tc::exp2_poly2(x[i], x[i]).x;
  }
}

}  // namespace
}  // namespace tb

extern "C" tb_status tb_diag_exp2(const float* x, float* y, int64_t n, tb_stream_t stream) {
  if (n < 0 || (n > 0 && (!x || !y))) return TB_ERR_INVALID_ARG;
  if (n == 0) return TB_OK;
  const int64_t pairs = (n + 1) / 2;
  const int64_t blocks = (pairs + 255) / 256;
  if (blocks > 0x7fffffff) return TB_ERR_UNSUPPORTED;
  tb::exp2_poly_kernel<<<(unsigned)blocks, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(x, y, n);
  tb::count_launches(1);
  return tb::cuda_status(cudaGetLastError());
}
