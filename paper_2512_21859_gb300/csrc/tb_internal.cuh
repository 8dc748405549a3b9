// Internal declarations shared by the kernels and the C-ABI layer.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "timebill_kv.h"

namespace tb {

// Bits of the device status word kept at the start of every workspace.
enum : int32_t {
  kStatusTimeout = 1,  // a bounded wait gave up
  kStatusRange = 2,    // a device-side range check fired
};

// Bytes reserved at the start of each workspace for the status word (word 0)
// and the grid-barrier counter of the fused scoring kernel (word
// kGridSyncWord); all of it is zeroed at the start of every call.
constexpr size_t kStatusBytes = 256;
constexpr int kGridSyncWord = 16;


// Largest G*W (window rows of one KV-head group) the scoring kernels take.
constexpr int kMaxWindowRows = 1024;

// Keys per work item of the SIMT scoring kernels.
constexpr int kSimtChunk = 256;

struct EvictReq {
  int64_t kv_off;     // first row of the request in K, V
  int64_t out_off;    // first row in Kc, Vc
  int64_t score_off;  // first column in scores / pooled
  int64_t idx_off;    // first column in idx
  int32_t n;          // prompt length N_b
  int32_t p;          // prefix length P_b = N_b - W
  int32_t k;          // retained prefix tokens k_b
  int32_t item0;      // first work item of the request in the scoring grid
};

struct EvictParams {
  int32_t batch, hq, hkv, group, d, window, pool_k, dtype;
  int32_t m_rows;     // G * W window rows per KV head
  int32_t chunk;      // keys per scoring work item
  int32_t items;      // total scoring work items
  int32_t max_p;      // max_b P_b
  int32_t max_r;      // max_b R_b
  int32_t flags;      // TB_EVICT_* bits of the descriptor
  int64_t kv_rows, out_rows, score_rows, idx_rows;
  float scale_log2;   // log2(e) / sqrt(d)
  float rowc_scale;   // c_row = rowc[r] * rowc_scale in log2 units: 1 for the
                      // library's own statistics, log2(e) for a caller's
                      // natural-log LSE (tb_window_scores_lse)
  EvictReq req[TB_MAX_BATCH];
};

struct DecodeParams {
  int32_t batch, hq, hkv, group, d, dtype, out_dtype, splits;
  int32_t split_len;  // keys per split
  // 1: the kernel just before the decode on the stream is the library's own
  // clearing kernel, so the first K/V tiles may be requested before the
  // dependency wait; 2: the same on the caller's word (prepared workspace
  // with TB_DECODE_EARLY_CACHE_READ) that the work before it writes no cache
  // row below lens[b] - 1, which is read again after the wait; 3
  // (TB_DECODE_CONCURRENT): no dependency wait before the work (the work
  // before it writes nothing the decode reads), one thread waits at the end
  // so that the grid still completes after it; 0 (prepared workspaces otherwise):
  // anything may precede it
  int32_t early_tma;
  int64_t cache_rows;
  int64_t max_len;
  float scale_log2;
  // 1: the split kernel leaves its partials and a merge kernel launched
  // behind it (programmatic dependent launch) merges them; 0: the last split
  // CTA of each (request, KV head) merges them, found with a split counter
  int32_t merge_kernel;
  int64_t cache_off[TB_MAX_BATCH];
  int32_t cache_cap[TB_MAX_BATCH];
};

// Workspace carving for the decode call (byte offsets, 256-aligned).
struct DecodeWorkspace {
  size_t status, counters, part_o, part_ml, total;  // [0, part_o) is zeroed per call
};

// Validates a decode descriptor and fills the kernel parameters.
tb_status build_decode(const tb_decode_desc* d, DecodeParams* p);
// Byte layout of the decode workspace for validated parameters.
DecodeWorkspace carve_decode(const DecodeParams& p);
// Maps a CUDA error to a status, keeping its text for tb_last_error_detail.
tb_status cuda_status(cudaError_t e);

// Workspace carving for the eviction calls (byte offsets, 256-aligned).
// status: kStatusBytes; tilectr: two tile counters per (request, KV head) of
// the tensor-core scoring kernel; lsum: fp64 row sums sum_c l_c 2^(m_c) of
// its window rows; [0, zeroed) is cleared by every call.
struct EvictWorkspace {
  size_t status, tilectr, lsum, zeroed, scores, partial, rowc, pooled, total;
};

// 2-D bf16 TMA map over rows of d elements, boxes of box_rows x 64 columns
// with 128-byte swizzle; false if the driver entry point is missing.
bool make_bf16_map(CUtensorMap* map, const void* base, int d, uint64_t rows, int box_rows);

// Adds n to the process-wide launch counter (tb_launch_counter).
void count_launches(int n);

struct NvtxRange {
  explicit NvtxRange(const char* name);
  ~NvtxRange();
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Programmatic dependent launch. A kernel launched by launch_pdl may begin
// (its CTAs made resident, their set-up run) while the previous kernel of the
// stream is still finishing: it calls pdl_wait() before its first access to
// global memory, which returns once that kernel has completed and its writes
// are visible, and pdl_trigger() after it, which lets the next such launch
// start early. Both are no-ops for a kernel launched the ordinary way.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// False when the environment sets TB_NO_PDL (ordinary launches throughout).
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

// Zeroes the first `bytes` (a multiple of 16) of a workspace on stream s
// with one small kernel.
cudaError_t clear_control_words(void* ws, size_t bytes, cudaStream_t s);

// ---------------------------------------------------------------------------
// launchers (each returns cudaGetLastError() of its launch)
// ---------------------------------------------------------------------------
cudaError_t launch_window_scores(const EvictParams& p, const void* q_win, const void* K,
                                 float* scores, float2* partial, float* rowc,
                                 int32_t* status, int32_t* tilectr, double* lsum, cudaStream_t s);
// The normalised window sums alone, from given per-row log2-sum-exp values
// (rowc [B][Hkv][G*W], scaled by p.rowc_scale): one QK^T pass.
cudaError_t launch_window_votes(const EvictParams& p, const void* q_win, const void* K,
                                float* scores, const float* rowc, int32_t* status,
                                int32_t* tilectr, cudaStream_t s);
cudaError_t launch_window_scores_simt(const EvictParams& p, const void* q_win, const void* K,
                                      float* scores, float2* partial, float* rowc,
                                      cudaStream_t s);
// Merges per-chunk (max, sum) partials into one log2-sum-exp per window row.
cudaError_t launch_window_combine(const EvictParams& p, const float2* partial, float* rowc,
                                  cudaStream_t s);
// Tensor-core scoring path (bf16, d in {64, 128}, G*W <= 256).
bool window_scores_tc_supported(const EvictParams& p);
// Whether the scoring kernel uses the fp64 row sums (workspace `lsum`) for
// some (request, KV head) of this descriptor; they are cleared only then.
bool window_scores_row_sums(const EvictParams& p);
cudaError_t launch_window_votes_tc(const EvictParams& p, const void* q_win, const void* K,
                                   float* scores, const float* rowc, int32_t* status,
                                   int32_t* tilectr, cudaStream_t s);
cudaError_t launch_window_votes_simt(const EvictParams& p, const void* q_win, const void* K,
                                     float* scores, const float* rowc, cudaStream_t s);
cudaError_t launch_window_scores_tc(const EvictParams& p, const void* q_win, const void* K,
                                    float* scores, float2* partial, float* rowc, int32_t* status,
                                    int32_t* tilectr, double* lsum, cudaStream_t s);
cudaError_t launch_pool(const EvictParams& p, const float* scores, float* pooled,
                        cudaStream_t s);
cudaError_t launch_select(const EvictParams& p, const float* pooled, int32_t* idx,
                          int32_t* status, cudaStream_t s);
// Cluster select with the max-pool fused in (pooled_out may be null).
constexpr int kClusterSliceMax = 16 * 1024;  // keys per CTA: 16 per thread of 1024
int select_cluster_size(const EvictParams& p);
bool select_cluster_supported(const EvictParams& p);
cudaError_t launch_select_cluster(const EvictParams& p, const float* scores, float* pooled_out,
                                  int32_t* idx, int32_t* status, cudaStream_t s);
// status may be null (tb_gather_kv has no workspace)
cudaError_t launch_gather(const EvictParams& p, const int32_t* idx, const void* K,
                          const void* V, void* Kc, void* Vc, int32_t* status, cudaStream_t s);
// TMA-staged bf16 decode (split partials only; the caller launches the combine).
bool decode_tma_supported(const DecodeParams& p);
cudaError_t launch_decode_tma(const DecodeParams& p, const void* q, const void* Kc,
                              const void* Vc, const int32_t* lens, float* part_o,
                              float2* part_ml, int32_t* counters, void* out, int32_t* status,
                              cudaStream_t s);
cudaError_t launch_decode(const DecodeParams& p, const void* q, const void* Kc,
                          const void* Vc, const int32_t* lens, void* out, float* part_o,
                          float2* part_ml, int32_t* counters, int32_t* status, cudaStream_t s);

// ---------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------
// Debug builds (TB_DEBUG=1, libtimebill_kv_debug.so) check invariants the
// release kernels take for granted (index ranges, finite normalisers, the
// selected count) and raise kStatusRange in the status word when one fails,
// instead of trapping; release builds compile the checks out.
#ifndef TB_DEBUG
#define TB_DEBUG 0
#endif
__device__ __forceinline__ void debug_flag(bool bad, int32_t* status) {
#if TB_DEBUG
  if (bad && status) atomicOr(status, kStatusRange);
#else
  (void)bad;
  (void)status;
#endif
}
__device__ __forceinline__ float bf16_bits_to_float(uint16_t v) {
  return __uint_as_float(static_cast<uint32_t>(v) << 16);
}

// fp32 -> bf16 bits, round to nearest even (NaN stays NaN).
__device__ __forceinline__ uint16_t float_to_bf16_rne(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7f800000u) == 0x7f800000u)
    return static_cast<uint16_t>((u >> 16) | ((u & 0xffffu) ? 0x40u : 0u));
  u += 0x7fffu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<uint16_t>(uint16_t v) { return bf16_bits_to_float(v); }

}  // namespace tb
