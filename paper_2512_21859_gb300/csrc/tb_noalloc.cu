// Decode attention for callers that may not allocate device memory.
//
// Some callers of a decode step cannot hand the library a workspace: a
// hard-real-time serving loop that forbids allocator calls on its per-token
// path (cudaMalloc can synchronise the device and take unbounded time, which
// a deadline-bound job cannot afford), or a plugin living inside a host
// framework that owns all device memory and exposes no allocator to it.
// tb_decode_attn_noalloc serves them: it runs the same split-K decode kernels
// as tb_decode_attn, but their scratch (split partials and the status word)
// lives in one file-scope device array of TB_NOALLOC_SCRATCH_BYTES that every
// GPU loading this library holds until the process exits.
//
// The array's host-side name is only a stand-in, never a device address: the
// first call on each device, with that device current, looks up the array's
// device address with cudaGetSymbolAddress and keeps it for later calls.
#include <cuda_runtime.h>

#include <mutex>

#include "tb_internal.cuh"

namespace tb {
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[TB_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once).
tb_status scratch_address(void** out) {
  int dev = -1;
  tb_status st = cuda_status(cudaGetDevice(&dev));
  if (st != TB_OK) return st;
  if (dev < 0 || dev >= kMaxDevices) return TB_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    st = cuda_status(cudaGetSymbolAddress(&p, g_noalloc_scratch));
    if (st != TB_OK) return st;
    if (p == nullptr) return TB_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return TB_OK;
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace
}  // namespace tb

using namespace tb;

extern "C" tb_status tb_decode_attn_noalloc(const tb_decode_desc* desc, const void* q,
                                            const void* Kc, const void* Vc, const int32_t* lens,
                                            void* out, tb_stream_t stream) {
  DecodeParams p;
  tb_status st = build_decode(desc, &p);
  if (st != TB_OK) return st;
  if (!q || !Kc || !Vc || !lens || !out) return TB_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(Kc) || !aligned16(Vc) || !aligned16(out))
    return TB_ERR_INVALID_ARG;
  const DecodeWorkspace w = carve_decode(p);
  if (w.total > (size_t)TB_NOALLOC_SCRATCH_BYTES) return TB_ERR_WORKSPACE;
  void* ws = nullptr;
  if ((st = scratch_address(&ws)) != TB_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(ws);
  // the split partials are fully rewritten by every call; the status word and
  // the split counters (everything before the partials) must start at zero
  if ((st = cuda_status(clear_control_words(base, w.part_o, s))) != TB_OK) return st;
  return cuda_status(launch_decode(p, q, Kc, Vc, lens, out,
                                   reinterpret_cast<float*>(base + w.part_o),
                                   reinterpret_cast<float2*>(base + w.part_ml),
                                   reinterpret_cast<int32_t*>(base + w.counters),
                                   reinterpret_cast<int32_t*>(base + w.status), s));
}
