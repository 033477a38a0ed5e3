// C-ABI entry points of libsgdkv: argument checks, workspace carving, launches.
#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "sgdkv_internal.cuh"

namespace sgdkv {

namespace {
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

namespace {
std::atomic<uint64_t> g_launches{0};
}  // namespace

void note_launches(int n) { g_launches.fetch_add(uint64_t(n), std::memory_order_relaxed); }

WsLayout workspace_layout(int32_t Hkv, int64_t L) {
  WsLayout w{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  const size_t H = size_t(Hkv);
  w.status = take(kStatusRegionBytes);
  w.partial = take(H * size_t(kMaxScoreParts) * kMaxRows * sizeof(float2));
  w.raw = take(4 * H * size_t(L) * sizeof(float));
  w.pooled = take(H * size_t(L) * sizeof(float));
  w.total = off;
  return w;
}

Ws workspace_view(void* base, const WsLayout& lay) {
  char* b = static_cast<char*>(base);
  Ws ws;
  ws.status = reinterpret_cast<uint32_t*>(b + lay.status);
  ws.sched = reinterpret_cast<uint32_t*>(b + lay.status + kSchedOffset);
  ws.partial = reinterpret_cast<float2*>(b + lay.partial);
  ws.raw = reinterpret_cast<float*>(b + lay.raw);
  ws.pooled = reinterpret_cast<float*>(b + lay.pooled);
  return ws;
}

namespace {

// Shape limits of v1 (see sgdkv.h).  Returns SGDKV_OK or the error to report.
sgdkv_status check_score_shape(int32_t Hq, int32_t Hkv, int64_t L, int32_t d, int32_t W) {
  if (Hq <= 0 || Hkv <= 0 || L <= 0 || d <= 0 || W <= 0) return SGDKV_ERR_INVALID_ARG;
  if (Hq % Hkv != 0 || W > L) return SGDKV_ERR_INVALID_ARG;
  if (d != kD || Hkv > SGDKV_MAX_KV_HEADS) return SGDKV_ERR_UNSUPPORTED;
  const int64_t GW = int64_t(Hq / Hkv) * W;
  if (GW > kMaxRows || GW % 32 != 0) return SGDKV_ERR_UNSUPPORTED;
  if (int64_t(Hkv) * L >= (int64_t(1) << 31)) return SGDKV_ERR_UNSUPPORTED;
  return SGDKV_OK;
}

sgdkv_status check_workspace(void* ws, size_t ws_bytes, int32_t Hkv, int64_t L) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SGDKV_ERR_WORKSPACE;
  if (ws_bytes < workspace_layout(Hkv, L).total) return SGDKV_ERR_WORKSPACE;
  return SGDKV_OK;
}

constexpr size_t kDecodePartOffset = 256;   // decode workspace: status word, then partials

sgdkv_status check_pool(int32_t pool) {
  if (pool < 1 || pool > 63 || pool % 2 == 0) return SGDKV_ERR_INVALID_ARG;
  return SGDKV_OK;
}

// Steps a4-a6 from the raw planes of the scoring workspace sws: the max-pool inside the
// selection kernel where its slices stay in registers, else the stand-alone pool kernel
// into scores_out followed by the selection on scores_out.  Device errors go to ws.
cudaError_t pool_then_compact(const Ws& sws, int32_t pool, uint32_t flags,
                              const __nv_bfloat16* K, const __nv_bfloat16* V, const HeadTable& ht,
                              int64_t total, float* scores_out, int32_t* indices_out,
                              int32_t* cu_out, __nv_bfloat16* K_out, __nv_bfloat16* V_out,
                              const Ws& ws, cudaStream_t st) {
  if (compact_pools_inline(ht.L)) {
    PoolSrc ps;
    ps.raw = sws.raw;
    ps.plane = int64_t(ht.Hkv) * ht.L;
    ps.radius = pool / 2;
    ps.combine_max = (flags & SGDKV_SCORE_AGG_MASK) == SGDKV_SCORE_AGG_IPT_MAX ? 1 : 0;
    ps.out = scores_out;
    return launch_compact(K, V, scores_out, ht, indices_out, cu_out, K_out, V_out, total, ws, st,
                          &ps);
  }
  cudaError_t e = launch_pool(sws, ht.Hkv, ht.L, pool, flags, scores_out, st);
  if (e != cudaSuccess) return e;
  return launch_compact(K, V, scores_out, ht, indices_out, cu_out, K_out, V_out, total, ws, st);
}

// Validates budgets and fills the per-head table; returns the total kept rows.
sgdkv_status build_head_table(const int64_t* budgets, int32_t Hkv, int64_t L, int64_t n_sink,
                              int64_t n_recent, HeadTable* ht, int64_t* total) {
  if (!budgets) return SGDKV_ERR_INVALID_ARG;
  if (n_sink < 0 || n_recent < 0 || n_sink + n_recent > L) return SGDKV_ERR_INVALID_ARG;
  std::memset(ht, 0, sizeof(*ht));
  ht->Hkv = Hkv;
  ht->L = L;
  ht->n_sink = n_sink;
  ht->n_recent = n_recent;
  int64_t acc = 0;
  ht->cu[0] = 0;
  for (int h = 0; h < Hkv; ++h) {
    const int64_t b = budgets[h];
    if (b < n_sink + n_recent || b > L) return SGDKV_ERR_INVALID_ARG;
    ht->k_mid[h] = int32_t(b - n_sink - n_recent);
    acc += b;
    ht->cu[h + 1] = int32_t(acc);
  }
  *total = acc;
  return SGDKV_OK;
}

thread_local cudaError_t t_last_cuda = cudaSuccess;

sgdkv_status from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return SGDKV_OK;
  t_last_cuda = e;
  return SGDKV_ERR_CUDA;
}

}  // namespace
}  // namespace sgdkv

using namespace sgdkv;

// ---------------------------------------------------------------------------------------
// Scratch for sgdkv_score_static: for callers that cannot allocate device memory
// themselves.  Lives in this file's module for as long as the library is loaded on a GPU.
// ---------------------------------------------------------------------------------------
static constexpr size_t kStaticScratchBytes = size_t(64) << 20;   // 64 MiB per device
static __device__ __align__(256) uint8_t sgdkv_static_scratch[kStaticScratchBytes];

namespace {
// Every scoring flag bit sgdkv.h defines.
constexpr uint32_t kScoreFlags =
    SGDKV_SCORE_PROXY_QUERY | SGDKV_SCORE_AGG_MASK | SGDKV_SCORE_DETERMINISTIC;

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_dev[kMaxDevices] = {};

// Device address of the static scratch on the current device (looked up once per device,
// with that device current; the host-side name is only a stand-in for it).
sgdkv_status static_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return from_cuda(e);
  if (dev < 0 || dev >= kMaxDevices) return SGDKV_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_dev[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, sgdkv_static_scratch);
    if (e != cudaSuccess) return from_cuda(e);
    g_scratch_dev[dev] = ptr;
  }
  *out = g_scratch_dev[dev];
  return SGDKV_OK;
}
}  // namespace

extern "C" {

const char* sgdkv_status_string(int status) {
  switch (status) {
    case SGDKV_OK: return "ok";
    case SGDKV_ERR_INVALID_ARG: return "invalid argument";
    case SGDKV_ERR_INFEASIBLE_BUDGET: return "infeasible budget";
    case SGDKV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
    case SGDKV_ERR_CUDA: return "CUDA error";
    case SGDKV_ERR_TIMEOUT: return "device-side wait timed out";
    case SGDKV_ERR_UNSUPPORTED: return "shape outside the supported limits";
    case SGDKV_ERR_INTERNAL: return "device-side consistency check failed";
    default: return "unknown status";
  }
}

int sgdkv_version(void) { return 100; }

uint64_t sgdkv_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char* sgdkv_last_cuda_error_string(void) { return cudaGetErrorString(t_last_cuda); }

void sgdkv_debug_set_score_hooks(uint32_t flags, uint64_t wait_ns) {
  g_score_flags = flags;
  g_score_wait_ns = wait_ns > 0 ? wait_ns : 2000000000ull;
}

size_t sgdkv_workspace_bytes(int32_t Hq, int32_t Hkv, int64_t L, int32_t d, int32_t W) {
  if (check_score_shape(Hq, Hkv, L, d, W) != SGDKV_OK) return 0;
  return workspace_layout(Hkv, L).total;
}

// Arguments of the scoring passes (sgdkv_score_ex, sgdkv_score_raw).
sgdkv_status check_score_args(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                              int64_t L, int32_t d, int32_t W, uint32_t flags,
                              const float* head_weights) {
  if (!q_win || !K) return SGDKV_ERR_INVALID_ARG;
  if (!aligned16(q_win) || !aligned16(K)) return SGDKV_ERR_INVALID_ARG;
  if (flags & ~kScoreFlags) return SGDKV_ERR_INVALID_ARG;
  const uint32_t agg = flags & SGDKV_SCORE_AGG_MASK;
  if (agg != SGDKV_SCORE_AGG_SUM && !head_weights) return SGDKV_ERR_INVALID_ARG;
  const sgdkv_status s = check_score_shape(Hq, Hkv, L, d, W);
  if (s != SGDKV_OK) return s;
  if (agg == SGDKV_SCORE_AGG_IPT_MAX && (W % 16 != 0 || W > 64 || Hq / Hkv > 8))
    return SGDKV_ERR_UNSUPPORTED;
  return SGDKV_OK;
}

sgdkv_status sgdkv_score_ex(const void* q_win, const void* K, int32_t Hq, int32_t Hkv, int64_t L,
                            int32_t d, int32_t W, int32_t pool, uint32_t flags,
                            const float* head_weights, float* scores_out, void* workspace,
                            size_t ws_bytes, void* stream) {
  if (!scores_out || !aligned16(scores_out)) return SGDKV_ERR_INVALID_ARG;
  sgdkv_status s = check_score_args(q_win, K, Hq, Hkv, L, d, W, flags, head_weights);
  if (s != SGDKV_OK) return s;
  if ((s = check_pool(pool)) != SGDKV_OK) return s;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  const uint32_t agg = flags & SGDKV_SCORE_AGG_MASK;
  return from_cuda(launch_score(static_cast<const __nv_bfloat16*>(q_win),
                                static_cast<const __nv_bfloat16*>(K), Hq, Hkv, L, W, pool, flags,
                                agg == SGDKV_SCORE_AGG_SUM ? nullptr : head_weights, scores_out,
                                ws, static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_score_raw(const void* q_win, const void* K, int32_t Hq, int32_t Hkv, int64_t L,
                             int32_t d, int32_t W, uint32_t flags, const float* head_weights,
                             void* workspace, size_t ws_bytes, void* stream) {
  sgdkv_status s = check_score_args(q_win, K, Hq, Hkv, L, d, W, flags, head_weights);
  if (s != SGDKV_OK) return s;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  const uint32_t agg = flags & SGDKV_SCORE_AGG_MASK;
  return from_cuda(launch_score_raw(static_cast<const __nv_bfloat16*>(q_win),
                                    static_cast<const __nv_bfloat16*>(K), Hq, Hkv, L, W, flags,
                                    agg == SGDKV_SCORE_AGG_SUM ? nullptr : head_weights, ws,
                                    static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_window_stats(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                                int64_t L, int32_t d, int32_t W, uint32_t flags,
                                const float* head_weights, void* workspace, size_t ws_bytes,
                                void* stream) {
  sgdkv_status s = check_score_args(q_win, K, Hq, Hkv, L, d, W, flags, head_weights);
  if (s != SGDKV_OK) return s;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  const uint32_t agg = flags & SGDKV_SCORE_AGG_MASK;
  return from_cuda(launch_passes(static_cast<const __nv_bfloat16*>(q_win),
                                 static_cast<const __nv_bfloat16*>(K), Hq, Hkv, L, W, flags,
                                 agg == SGDKV_SCORE_AGG_SUM ? nullptr : head_weights, ws,
                                 static_cast<cudaStream_t>(stream), 1u));
}

sgdkv_status sgdkv_window_sums(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                               int64_t L, int32_t d, int32_t W, uint32_t flags,
                               const float* head_weights, void* workspace, size_t ws_bytes,
                               void* stream) {
  sgdkv_status s = check_score_args(q_win, K, Hq, Hkv, L, d, W, flags, head_weights);
  if (s != SGDKV_OK) return s;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  const uint32_t agg = flags & SGDKV_SCORE_AGG_MASK;
  return from_cuda(launch_passes(static_cast<const __nv_bfloat16*>(q_win),
                                 static_cast<const __nv_bfloat16*>(K), Hq, Hkv, L, W, flags,
                                 agg == SGDKV_SCORE_AGG_SUM ? nullptr : head_weights, ws,
                                 static_cast<cudaStream_t>(stream), 2u));
}

sgdkv_status sgdkv_pool_raw(const void* workspace, size_t ws_bytes, int32_t Hkv, int64_t L,
                            int32_t pool, uint32_t flags, float* scores_out, void* stream) {
  if (!scores_out || !aligned16(scores_out)) return SGDKV_ERR_INVALID_ARG;
  if (Hkv <= 0 || L <= 0) return SGDKV_ERR_INVALID_ARG;
  if (Hkv > SGDKV_MAX_KV_HEADS || int64_t(Hkv) * L >= (int64_t(1) << 31))
    return SGDKV_ERR_UNSUPPORTED;
  if (flags & ~kScoreFlags) return SGDKV_ERR_INVALID_ARG;
  sgdkv_status s = check_pool(pool);
  if (s != SGDKV_OK) return s;
  if ((s = check_workspace(const_cast<void*>(workspace), ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(const_cast<void*>(workspace), workspace_layout(Hkv, L));
  return from_cuda(launch_pool(ws, Hkv, L, pool, flags, scores_out,
                               static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_score(const void* q_win, const void* K, int32_t Hq, int32_t Hkv, int64_t L,
                         int32_t d, int32_t W, int32_t pool, float* scores_out,
                         void* workspace, size_t ws_bytes, void* stream) {
  return sgdkv_score_ex(q_win, K, Hq, Hkv, L, d, W, pool, 0u, nullptr, scores_out, workspace,
                        ws_bytes, stream);
}

sgdkv_status sgdkv_score_static(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                                int64_t L, int32_t d, int32_t W, int32_t pool, float* scores_out,
                                uint32_t* status_out, void* stream) {
  if (!q_win || !K || !scores_out) return SGDKV_ERR_INVALID_ARG;
  if (!aligned16(q_win) || !aligned16(K) || !aligned16(scores_out)) return SGDKV_ERR_INVALID_ARG;
  sgdkv_status s = check_score_shape(Hq, Hkv, L, d, W);
  if (s != SGDKV_OK) return s;
  if ((s = check_pool(pool)) != SGDKV_OK) return s;
  // scoring uses the status word, the pass-1 partials and the raw planes: everything in
  // the workspace layout before the pooled-score scratch of sgdkv_compress_layer
  const WsLayout lay = workspace_layout(Hkv, L);
  if (lay.pooled > kStaticScratchBytes) return SGDKV_ERR_WORKSPACE;
  void* scratch = nullptr;
  if ((s = static_scratch(&scratch)) != SGDKV_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Ws ws = workspace_view(scratch, lay);
  // the status word and the scorer's tile counters start at zero
  cudaError_t e = cudaMemsetAsync(ws.status, 0, kStatusRegionBytes, st);
  if (e != cudaSuccess) return from_cuda(e);
  e = launch_score(static_cast<const __nv_bfloat16*>(q_win), static_cast<const __nv_bfloat16*>(K),
                   Hq, Hkv, L, W, pool, 0u, nullptr, scores_out, ws, st);
  if (e != cudaSuccess) return from_cuda(e);
  if (status_out) {
    e = cudaMemcpyAsync(status_out, ws.status, sizeof(uint32_t), cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return from_cuda(e);
  }
  return SGDKV_OK;
}

sgdkv_status sgdkv_compact(const void* K, const void* V, const float* scores,
                           const int64_t* budgets, int32_t Hkv, int64_t L, int32_t d,
                           int64_t n_sink, int64_t n_recent, int32_t* indices_out,
                           int32_t* cu_seqlens_out, void* K_out, void* V_out, void* workspace,
                           size_t ws_bytes, void* stream) {
  if (!K || !V || !scores || !cu_seqlens_out) return SGDKV_ERR_INVALID_ARG;
  if (Hkv <= 0 || L <= 0 || d <= 0) return SGDKV_ERR_INVALID_ARG;
  if (d != kD || Hkv > SGDKV_MAX_KV_HEADS || int64_t(Hkv) * L >= (int64_t(1) << 31))
    return SGDKV_ERR_UNSUPPORTED;
  if (!aligned16(K) || !aligned16(V) || !aligned16(scores)) return SGDKV_ERR_INVALID_ARG;
  HeadTable ht;
  int64_t total = 0;
  sgdkv_status s = build_head_table(budgets, Hkv, L, n_sink, n_recent, &ht, &total);
  if (s != SGDKV_OK) return s;
  if (total > 0 && (!indices_out || !K_out || !V_out)) return SGDKV_ERR_INVALID_ARG;
  if (total > 0 && (!aligned16(K_out) || !aligned16(V_out))) return SGDKV_ERR_INVALID_ARG;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  return from_cuda(launch_compact(static_cast<const __nv_bfloat16*>(K),
                                  static_cast<const __nv_bfloat16*>(V), scores, ht, indices_out,
                                  cu_seqlens_out, static_cast<__nv_bfloat16*>(K_out),
                                  static_cast<__nv_bfloat16*>(V_out), total, ws,
                                  static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_pool_compact(const void* score_workspace, size_t score_ws_bytes, int32_t pool,
                                uint32_t flags, const void* K, const void* V,
                                const int64_t* budgets, int32_t Hkv, int64_t L, int32_t d,
                                int64_t n_sink, int64_t n_recent, float* scores_out,
                                int32_t* indices_out, int32_t* cu_seqlens_out, void* K_out,
                                void* V_out, void* workspace, size_t ws_bytes, void* stream) {
  if (!K || !V || !scores_out || !cu_seqlens_out) return SGDKV_ERR_INVALID_ARG;
  if (Hkv <= 0 || L <= 0 || d <= 0) return SGDKV_ERR_INVALID_ARG;
  if (d != kD || Hkv > SGDKV_MAX_KV_HEADS || int64_t(Hkv) * L >= (int64_t(1) << 31))
    return SGDKV_ERR_UNSUPPORTED;
  if (!aligned16(K) || !aligned16(V) || !aligned16(scores_out)) return SGDKV_ERR_INVALID_ARG;
  if (flags & ~kScoreFlags) return SGDKV_ERR_INVALID_ARG;
  sgdkv_status s = check_pool(pool);
  if (s != SGDKV_OK) return s;
  HeadTable ht;
  int64_t total = 0;
  if ((s = build_head_table(budgets, Hkv, L, n_sink, n_recent, &ht, &total)) != SGDKV_OK) return s;
  if (total > 0 && (!indices_out || !K_out || !V_out)) return SGDKV_ERR_INVALID_ARG;
  if (total > 0 && (!aligned16(K_out) || !aligned16(V_out))) return SGDKV_ERR_INVALID_ARG;
  if ((s = check_workspace(const_cast<void*>(score_workspace), score_ws_bytes, Hkv, L)) != SGDKV_OK)
    return s;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws sws = workspace_view(const_cast<void*>(score_workspace), workspace_layout(Hkv, L));
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  return from_cuda(pool_then_compact(sws, pool, flags, static_cast<const __nv_bfloat16*>(K),
                                     static_cast<const __nv_bfloat16*>(V), ht, total, scores_out,
                                     indices_out, cu_seqlens_out,
                                     static_cast<__nv_bfloat16*>(K_out),
                                     static_cast<__nv_bfloat16*>(V_out), ws,
                                     static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_compress_layer(const void* q_win, const void* K, const void* V,
                                  const int64_t* budgets, int32_t Hq, int32_t Hkv, int64_t L,
                                  int32_t d, int32_t W, int32_t pool, int64_t n_sink,
                                  int64_t n_recent, float* scores_out, int32_t* indices_out,
                                  int32_t* cu_seqlens_out, void* K_out, void* V_out,
                                  void* workspace, size_t ws_bytes, void* stream) {
  if (!q_win || !K || !V || !cu_seqlens_out) return SGDKV_ERR_INVALID_ARG;
  if (!aligned16(q_win) || !aligned16(K) || !aligned16(V)) return SGDKV_ERR_INVALID_ARG;
  if (scores_out && !aligned16(scores_out)) return SGDKV_ERR_INVALID_ARG;
  sgdkv_status s = check_score_shape(Hq, Hkv, L, d, W);
  if (s != SGDKV_OK) return s;
  if ((s = check_pool(pool)) != SGDKV_OK) return s;
  HeadTable ht;
  int64_t total = 0;
  if ((s = build_head_table(budgets, Hkv, L, n_sink, n_recent, &ht, &total)) != SGDKV_OK) return s;
  if (total > 0 && (!indices_out || !K_out || !V_out)) return SGDKV_ERR_INVALID_ARG;
  if (total > 0 && (!aligned16(K_out) || !aligned16(V_out))) return SGDKV_ERR_INVALID_ARG;
  if ((s = check_workspace(workspace, ws_bytes, Hkv, L)) != SGDKV_OK) return s;
  const Ws ws = workspace_view(workspace, workspace_layout(Hkv, L));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* pooled = scores_out ? scores_out : ws.pooled;
  cudaError_t e = launch_score_raw(static_cast<const __nv_bfloat16*>(q_win),
                                   static_cast<const __nv_bfloat16*>(K), Hq, Hkv, L, W, 0u,
                                   nullptr, ws, st);
  if (e != cudaSuccess) return from_cuda(e);
  return from_cuda(pool_then_compact(ws, pool, 0u, static_cast<const __nv_bfloat16*>(K),
                                     static_cast<const __nv_bfloat16*>(V), ht, total, pooled,
                                     indices_out, cu_seqlens_out,
                                     static_cast<__nv_bfloat16*>(K_out),
                                     static_cast<__nv_bfloat16*>(V_out), ws, st));
}

size_t sgdkv_decode_workspace_bytes(int32_t Hq, int32_t Hkv, int32_t n_tok, int32_t d,
                                    int64_t total_rows) {
  if (Hq <= 0 || Hkv <= 0 || n_tok <= 0 || d != kD || total_rows < 0) return 0;
  if (Hq % Hkv != 0 || Hkv > SGDKV_MAX_KV_HEADS || (Hq / Hkv) * n_tok > 16) return 0;
  if (total_rows >= (int64_t(1) << 31)) return 0;
  return kDecodePartOffset + decode_partial_bytes(total_rows, Hkv);
}

sgdkv_status sgdkv_decode_attention(const void* q, int32_t Hq, int32_t Hkv, int32_t n_tok,
                                    int32_t d, const void* K_cache, const void* V_cache,
                                    const int64_t* budgets, float* out, void* workspace,
                                    size_t ws_bytes, void* stream) {
  if (!q || !budgets || !out) return SGDKV_ERR_INVALID_ARG;
  if (Hq <= 0 || Hkv <= 0 || n_tok <= 0 || d <= 0 || Hq % Hkv != 0) return SGDKV_ERR_INVALID_ARG;
  if (d != kD || Hkv > SGDKV_MAX_KV_HEADS || (Hq / Hkv) * n_tok > 16) return SGDKV_ERR_UNSUPPORTED;
  int64_t total = 0;
  for (int h = 0; h < Hkv; ++h) {
    if (budgets[h] < 0) return SGDKV_ERR_INVALID_ARG;
    total += budgets[h];
    if (total >= (int64_t(1) << 31)) return SGDKV_ERR_UNSUPPORTED;
  }
  if (total > 0 && (!K_cache || !V_cache)) return SGDKV_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || (total > 0 && (!aligned16(K_cache) || !aligned16(V_cache))))
    return SGDKV_ERR_INVALID_ARG;
  const size_t need = sgdkv_decode_workspace_bytes(Hq, Hkv, n_tok, d, total);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 || ws_bytes < need)
    return SGDKV_ERR_WORKSPACE;
  float* part = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + kDecodePartOffset);
  return from_cuda(launch_decode(static_cast<const __nv_bfloat16*>(q),
                                 static_cast<const __nv_bfloat16*>(K_cache),
                                 static_cast<const __nv_bfloat16*>(V_cache), budgets, Hq, Hkv,
                                 n_tok, out, part, ws_bytes - kDecodePartOffset,
                                 static_cast<cudaStream_t>(stream)));
}

sgdkv_status sgdkv_last_error(void* workspace, void* stream) {
  if (!workspace) return SGDKV_ERR_WORKSPACE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t code = 0;
  cudaError_t e;
  if ((e = cudaMemcpyAsync(&code, workspace, sizeof(code), cudaMemcpyDeviceToHost, st)) != cudaSuccess)
    return from_cuda(e);
  if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return from_cuda(e);
  if (code != 0) {
    const uint32_t zero = 0;
    if ((e = cudaMemcpyAsync(workspace, &zero, sizeof(zero), cudaMemcpyHostToDevice, st)) != cudaSuccess)
      return from_cuda(e);
    if ((e = cudaStreamSynchronize(st)) != cudaSuccess) return from_cuda(e);
  }
  return static_cast<sgdkv_status>(code);
}

}  // extern "C"
