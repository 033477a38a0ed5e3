// Internal declarations shared by the libsgdkv translation units (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "sgdkv.h"

namespace sgdkv {

constexpr int kD = SGDKV_HEAD_DIM;     // head dim supported by v1
constexpr int kMaxRows = 512;          // G*W limit (window rows of one KV head)
constexpr int kMaxScoreParts = 320;    // pass-1 partial (m, Z) slots per KV head
constexpr int kMaxPoolRadius = 31;     // max-pool window <= 63 positions
// Per-call, per-head constants passed by value in kernel parameters.
struct HeadTable {
  int32_t Hkv;
  int32_t pad0;
  int64_t L;
  int64_t n_sink;
  int64_t n_recent;
  int32_t cu[SGDKV_MAX_KV_HEADS + 1];   // cu_seqlens of the output
  int32_t k_mid[SGDKV_MAX_KV_HEADS];    // middle tokens to select: b_h - n_sink - n_recent
};

// Device views into the caller's workspace.
struct Ws {
  uint32_t* status;      // sticky first device-side error (sgdkv_status)
  uint32_t* sched;       // key-tile counters and finish counts of the two scoring passes
                         // (kSched* offsets; zero between launches)
  float2* partial;       // [Hkv][kMaxScoreParts][kMaxRows] per-CTA (max, sum), log2 units
  float* raw;            // [4][Hkv][L] window scores before pooling, as four partial sums
  float* pooled;         // [Hkv][L] pooled scores (compress_layer scratch)
};

struct WsLayout {
  size_t status, partial, raw, pooled, total;   // status region: status word, then sched
};
constexpr size_t kSchedOffset = 1024;           // byte offset of Ws::sched in the status region
// Ws::sched words: per head, the key-tile counters and finish counts of the two passes.
constexpr int kSchedPass1Tiles = 0;
constexpr int kSchedPass1Done = SGDKV_MAX_KV_HEADS;
constexpr int kSchedPass2Tiles = 2 * SGDKV_MAX_KV_HEADS;
constexpr int kSchedPass2Done = 3 * SGDKV_MAX_KV_HEADS;
constexpr size_t kStatusRegionBytes = kSchedOffset + 4 * SGDKV_MAX_KV_HEADS * sizeof(uint32_t);

__host__ __device__ inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

WsLayout workspace_layout(int32_t Hkv, int64_t L);
Ws workspace_view(void* base, const WsLayout& lay);

__device__ __forceinline__ void record_error(uint32_t* status, uint32_t code) {
  atomicCAS(status, 0u, code);
}

// Counts kernel launches issued by the library (sgdkv_launch_count).
void note_launches(int n);

// Brackets one kernel launch with CUDA events when kernel timing is enabled.
class KernelTimer {
 public:
  KernelTimer(int kind, cudaStream_t stream);
  ~KernelTimer();
  KernelTimer(const KernelTimer&) = delete;
  KernelTimer& operator=(const KernelTimer&) = delete;

 private:
  int kind_;
  cudaStream_t stream_;
  void* start_ = nullptr;
};

// Scorer wait bound and test-hook flags (sgdkv_debug_set_score_hooks).
extern uint64_t g_score_wait_ns;
extern uint32_t g_score_flags;

// Launchers (each returns cudaGetLastError() after its launches).
// flags: SGDKV_SCORE_* (0: the causal observation window of sgdkv_score, summed over the
// GQA group); head_weights: device fp32 [Hq] for the IPT aggregation modes, else NULL.
cudaError_t launch_score(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                         int64_t L, int W, int pool, uint32_t flags, const float* head_weights,
                         float* scores_out, const Ws& ws, cudaStream_t stream);
// The two halves of launch_score: both scoring passes into the raw planes of ws, and the
// max-pool of those planes into scores_out (flags select the planes' combination).
cudaError_t launch_score_raw(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                             int64_t L, int W, uint32_t flags, const float* head_weights,
                             const Ws& ws, cudaStream_t stream);
cudaError_t launch_pool(const Ws& ws, int Hkv, int64_t L, int pool, uint32_t flags,
                        float* scores_out, cudaStream_t stream);
// launch_score_raw's passes one at a time: bit 0 pass 1 (window-row statistics into the
// workspace), bit 1 pass 2 (the window sums, reading those statistics).
cudaError_t launch_passes(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                          int64_t L, int W, uint32_t flags, const float* head_weights,
                          const Ws& ws, cudaStream_t stream, unsigned passes);
// Source of the pooled scores when the selection kernel forms them itself: the four raw
// planes [4][Hkv][L] of a scoring workspace (plane stride `plane` floats), the window radius,
// the planes' combination (sum, or max for the "Ipt." max aggregation), and the output
// [Hkv][L] that receives the pooled scores the selection ran on.
struct PoolSrc {
  const float* raw;
  int64_t plane;
  int radius;
  int combine_max;
  float* out;
};
// pool_src NULL: select on `scores`.  Else `scores` is ignored and the selection kernel
// pools pool_src's planes first (only for rows that compact_pools_inline accepts).
cudaError_t launch_compact(const __nv_bfloat16* K, const __nv_bfloat16* V,
                           const float* scores, const HeadTable& ht, int32_t* indices_out,
                           int32_t* cu_out, __nv_bfloat16* K_out, __nv_bfloat16* V_out,
                           int64_t total_rows, const Ws& ws, cudaStream_t stream,
                           const PoolSrc* pool_src = nullptr);
// true when the selection kernel for rows of length L keeps its slice in registers, and so
// can take a PoolSrc
bool compact_pools_inline(int64_t L);

// Decode attention over the flat compressed cache (decode.cu): bytes of the per-warp
// partials for total_rows kept rows, and the launcher (q [Hq][T][128], K/V cache
// [sum b_h][128], out fp32 [Hq][T][128]; budgets on the host).
size_t decode_partial_bytes(int64_t total_rows, int Hkv);
cudaError_t launch_decode(const __nv_bfloat16* q, const __nv_bfloat16* Kc,
                          const __nv_bfloat16* Vc, const int64_t* budgets, int Hq, int Hkv,
                          int T, float* out, float* part, size_t part_bytes,
                          cudaStream_t stream);

}  // namespace sgdkv
