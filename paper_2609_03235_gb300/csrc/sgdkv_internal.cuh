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
constexpr int kSelChunk = 4096;        // selection elements per CTA
constexpr int kSelThreads = 256;       // threads per selection CTA (16 elements each)
constexpr int kSelPerThread = kSelChunk / kSelThreads;
constexpr int kRadixBins = 256;        // radix digit: 8 bits

// Per-head state of the radix selection (lives in the workspace).
struct SelState {
  uint32_t prefix;      // high bits of the threshold fixed so far
  uint32_t k_rem;       // elements still to take among those matching `prefix`
  uint32_t tau;         // final threshold (fp32 bit pattern of a non-negative score)
  uint32_t tie_quota;   // how many elements equal to tau are kept (lowest positions first)
  uint32_t pad[4];
};

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

// Device views into the caller's workspace.  The control block (status, histograms,
// counters, selection state) sits at fixed offsets sized for SGDKV_MAX_KV_HEADS, so the
// kernels that leave it cleared keep it valid for the next call whatever its shape.
struct Ws {
  uint32_t* status;      // sticky first device-side error (sgdkv_status)
  uint32_t* hist;        // [SGDKV_MAX_KV_HEADS][kRadixBins] radix histograms (kept zero)
  uint32_t* sel_cnt;     // [SGDKV_MAX_KV_HEADS] radix-pass completion counters (kept zero)
  SelState* sel;         // [SGDKV_MAX_KV_HEADS]
  uint2* chunk_cnt;      // [Hkv][n_sel_chunks] (kept non-ties, ties) per selection chunk
  float2* partial;       // [Hkv][kMaxScoreParts][kMaxRows] per-CTA (max, sum), log2 units
  float* raw;            // [4][Hkv][L] window scores before pooling, as four partial sums
  float* pooled;         // [Hkv][L] pooled scores (compress_layer scratch)
};

struct WsLayout {
  size_t status, hist, sel_cnt, sel, chunk_cnt, partial, raw, pooled, total;
};

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

WsLayout workspace_layout(int32_t Hkv, int64_t L);
Ws workspace_view(void* base, const WsLayout& lay);

__device__ __forceinline__ void record_error(uint32_t* status, uint32_t code) {
  atomicCAS(status, 0u, code);
}

// Counts kernel launches issued by the library (sgdkv_launch_count).
void note_launches(int n);

// Scorer wait bound and test-hook flags (sgdkv_debug_set_score_hooks).
extern uint64_t g_score_wait_ns;
extern uint32_t g_score_flags;

// Launchers (each returns cudaGetLastError() after its launches).
cudaError_t launch_score(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                         int64_t L, int W, int pool, float* scores_out, const Ws& ws,
                         cudaStream_t stream);
cudaError_t launch_compact(const __nv_bfloat16* K, const __nv_bfloat16* V,
                           const float* scores, const HeadTable& ht, int32_t* indices_out,
                           int32_t* cu_out, __nv_bfloat16* K_out, __nv_bfloat16* V_out,
                           int64_t total_rows, const Ws& ws, cudaStream_t stream);

}  // namespace sgdkv
