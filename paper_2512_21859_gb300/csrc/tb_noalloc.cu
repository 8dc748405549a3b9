// Decode attention for callers that may not allocate device memory.
//
// Some callers of a decode step cannot hand the library a workspace: a
// hard-real-time serving loop that forbids allocator calls on its per-token
// path (cudaMalloc can synchronise the device and take unbounded time, which
// a deadline-bound job cannot afford), or a plugin living inside a host
// framework that owns all device memory and exposes no allocator to it.
// tb_decode_attn_noalloc serves them: it runs the same split-K decode kernels
// as tb_decode_attn, but their scratch (split partials, split counters and
// the status word) lives in one file-scope device array of
// TB_NOALLOC_SCRATCH_BYTES that every GPU loading this library holds until
// the process exits.
//
// The array's host-side name is only a stand-in, never a device address: the
// first call in each CUDA context, with that context current, looks up the
// array's device address with cudaGetSymbolAddress and keeps it for later
// calls in the same context. The context is told apart by its unique id
// (cuCtxGetId), so a context created after cudaDeviceReset, or a driver-API
// context of the caller's own (where the module, and with it the array, has
// another address), gets its own lookup.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>

#include "tb_internal.cuh"

namespace tb {
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[TB_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

struct ScratchSlot {
  unsigned long long ctx_id;  // unique id of the context the address belongs to
  bool have_id;
  void* addr;
};

std::mutex g_scratch_mu;
ScratchSlot g_slot[kMaxDevices] = {};

// Driver entry points for the current context and its unique id (null when
// the driver lacks them; the cache is then kept per device only).
void context_fns(CtxGetCurrentFn* cur, CtxGetIdFn* id) {
  static CtxGetCurrentFn f_cur = nullptr;
  static CtxGetIdFn f_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f_cur = reinterpret_cast<CtxGetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f_id = reinterpret_cast<CtxGetIdFn>(f);
  });
  *cur = f_cur;
  *id = f_id;
}

// Unique id of the current context; false if there is none yet or the driver
// cannot say.
bool current_context_id(unsigned long long* out) {
  CtxGetCurrentFn cur;
  CtxGetIdFn idf;
  context_fns(&cur, &idf);
  if (!cur || !idf) return false;
  CUcontext ctx = nullptr;
  if (cur(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
  return idf(ctx, out) == CUDA_SUCCESS;
}

// Device address of the scratch array in the current context (looked up on
// the first call in each context, then kept).
tb_status scratch_address(void** out) {
  int dev = -1;
  tb_status st = cuda_status(cudaGetDevice(&dev));
  if (st != TB_OK) return st;
  if (dev < 0 || dev >= kMaxDevices) return TB_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  ScratchSlot& slot = g_slot[dev];
  unsigned long long id = 0;
  const bool have_id = current_context_id(&id);
  if (slot.addr != nullptr && (have_id ? (slot.have_id && slot.ctx_id == id) : !slot.have_id)) {
    *out = slot.addr;
    return TB_OK;
  }
  void* p = nullptr;
  st = cuda_status(cudaGetSymbolAddress(&p, g_noalloc_scratch));
  if (st != TB_OK) return st;
  if (p == nullptr) return TB_ERR_CUDA;
  // the lookup above makes the runtime's context current if none was
  slot.have_id = current_context_id(&slot.ctx_id);
  slot.addr = p;
  *out = p;
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

extern "C" tb_status tb_decode_noalloc_status(tb_stream_t stream, int32_t* raw) {
  void* ws = nullptr;
  tb_status st = scratch_address(&ws);
  if (st != TB_OK) return st;
  return tb_read_status(ws, TB_NOALLOC_SCRATCH_BYTES, stream, raw);
}
