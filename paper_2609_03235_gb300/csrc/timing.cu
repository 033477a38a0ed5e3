// Optional per-kernel timing (diagnostics): CUDA events recorded around every kernel the
// library launches, on the launch stream, while timing is enabled.  Launches captured into a
// CUDA graph are bracketed by event-record nodes of that graph; their records are read after
// the graph has run (one record per captured launch).
#include <mutex>
#include <vector>

#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace {
struct Record {
  int kind;
  cudaEvent_t start, end;
};
std::mutex g_mu;
uint32_t g_mask = 0;    // bit k: time kernels of kind k
std::vector<Record> g_pending;
std::vector<cudaEvent_t> g_free;

cudaEvent_t take_event() {
  if (!g_free.empty()) {
    cudaEvent_t e = g_free.back();
    g_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Records e on the stream; while the stream is being captured into a CUDA graph the record
// becomes an event-record node of the graph (taken each time the graph is launched).
void record(cudaEvent_t e, cudaStream_t stream) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(stream, &cs);
  if (cs == cudaStreamCaptureStatusActive) cudaEventRecordWithFlags(e, stream, cudaEventRecordExternal);
  else cudaEventRecord(e, stream);
}
}  // namespace

KernelTimer::KernelTimer(int kind, cudaStream_t stream) : kind_(kind), stream_(stream) {
  std::lock_guard<std::mutex> lock(g_mu);
  if (kind_ < 0 || kind_ >= SGDKV_KERNEL_KINDS || !(g_mask & (1u << kind_))) return;
  start_ = take_event();
  if (start_) record(static_cast<cudaEvent_t>(start_), stream_);
}

KernelTimer::~KernelTimer() {
  if (!start_) return;
  std::lock_guard<std::mutex> lock(g_mu);
  cudaEvent_t end = take_event();
  if (!end) {
    g_free.push_back(static_cast<cudaEvent_t>(start_));
    return;
  }
  record(end, stream_);
  g_pending.push_back(Record{kind_, static_cast<cudaEvent_t>(start_), end});
}

}  // namespace sgdkv

using namespace sgdkv;

extern "C" {

void sgdkv_debug_enable_kernel_timing(uint32_t kind_mask) {
  std::lock_guard<std::mutex> lock(g_mu);
  g_mask = kind_mask;
}

sgdkv_status sgdkv_debug_kernel_timing(int kind, double* total_ms, int64_t* launches) {
  if (!total_ms || !launches || kind < 0 || kind >= SGDKV_KERNEL_KINDS) return SGDKV_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lock(g_mu);
  double sum = 0.0;
  int64_t n = 0;
  std::vector<Record> keep;
  for (const Record& r : g_pending) {
    if (r.kind != kind) {
      keep.push_back(r);
      continue;
    }
    float ms = 0.f;
    if (cudaEventSynchronize(r.end) != cudaSuccess ||
        cudaEventElapsedTime(&ms, r.start, r.end) != cudaSuccess)
      return SGDKV_ERR_CUDA;
    sum += ms;
    ++n;
    g_free.push_back(r.start);
    g_free.push_back(r.end);
  }
  g_pending.swap(keep);
  *total_ms = sum;
  *launches = n;
  return SGDKV_OK;
}

}  // extern "C"
