// Token selection, ordered compaction and K/V gather (Section 3.3: keep sink and recent
// tokens, then each head's top (b_h - n_sink - n_recent) middle tokens by score; equal
// scores are broken by the lower position).
//
// Scores are finite and non-negative, so their fp32 bit patterns sort like their values
// and the threshold search is an exact most-significant-digit radix select on uint32 keys:
// four passes of 8-bit digits, each a histogram over the keys that match the digits fixed
// so far.  The CTA that finishes a pass last (atomic completion counter,
// no waiting) picks the next digit and clears the histogram for the next pass or call.  Compaction then keeps every middle key above the threshold tau plus the first
// `tie_quota` keys equal to tau in position order, and writes kept positions ascending.
#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace {

__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

// Exclusive scan of one value per thread over a CTA of kSelThreads threads.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* s_warp,
                                                    uint32_t* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  if (lane == 31) s_warp[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    const uint32_t x = lane < kSelThreads / 32 ? s_warp[lane] : 0u;
    const uint32_t xi = warp_incl_scan(x);
    if (lane < kSelThreads / 32) s_warp[lane] = xi - x;
    if (lane == kSelThreads / 32 - 1) s_warp[kSelThreads / 32] = xi;
  }
  __syncthreads();
  const uint32_t r = s_warp[wid] + incl - v;
  *total = s_warp[kSelThreads / 32];
  __syncthreads();
  return r;
}

// One 8-bit digit (bits 24-31, 16-23, 8-15, 0-7 in passes 0..3) of the radix select over
// the middle range of every head.  Each warp counts into its own shared-memory histogram
// (neighbouring positions have similar scores, so lanes of a warp often share a bin; the
// contention stays inside the warp), then the CTA adds its counts to the head's global
// histogram.
__global__ void __launch_bounds__(kSelThreads)
sel_radix_kernel(const float* __restrict__ scores, HeadTable ht, Ws ws, int pass, int nchunks) {
  constexpr int kWarps = kSelThreads / 32;
  const int h = blockIdx.y, c = blockIdx.x, tid = threadIdx.x, wid = tid >> 5;
  if (ht.k_mid[h] == 0) return;   // nothing to select from the middle of this head
  __shared__ uint32_t hist[kWarps][kRadixBins];
  __shared__ uint32_t s_warp[kWarps + 1];
  __shared__ int s_last;
  for (int i = tid; i < kWarps * kRadixBins; i += blockDim.x) (&hist[0][0])[i] = 0u;
  __syncthreads();
  const int shift = 24 - 8 * pass;
  const uint32_t prefix = pass == 0 ? 0u : ws.sel[h].prefix;
  const uint32_t hi_mask = pass == 0 ? 0u : (0xffffffffu << (32 - 8 * pass));
  const int64_t L = ht.L, mid_lo = ht.n_sink, mid_hi = ht.L - ht.n_recent;
  const int64_t beg = mid_lo + int64_t(c) * kSelChunk;
  const int64_t end = beg + kSelChunk < mid_hi ? beg + kSelChunk : mid_hi;
  const float* row = scores + int64_t(h) * L;
  for (int64_t j = beg + tid; j < end; j += blockDim.x) {
    const uint32_t u = __float_as_uint(__ldg(row + j));
    if ((u & hi_mask) == prefix) atomicAdd(&hist[wid][(u >> shift) & 255u], 1u);
  }
  __syncthreads();
  uint32_t* ghist = ws.hist + int64_t(h) * kRadixBins;
  {
    uint32_t cnt = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) cnt += hist[w][tid];
    if (cnt) atomicAdd(&ghist[tid], cnt);
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(&ws.sel_cnt[h], 1u) == uint32_t(nchunks - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // Last CTA of this head: thread t holds bin 255 - t (descending digit order).
  const uint32_t k_rem = pass == 0 ? uint32_t(ht.k_mid[h]) : ws.sel[h].k_rem;
  const uint32_t cnt = __ldcg(&ghist[255 - tid]);
  uint32_t total;
  const uint32_t excl = block_excl_scan(cnt, s_warp, &total);
  if (excl < k_rem && excl + cnt >= k_rem) {             // exactly one thread
    SelState st;
    st.prefix = prefix | (uint32_t(255 - tid) << shift);
    st.k_rem = k_rem - excl;
    st.tau = st.prefix;
    st.tie_quota = st.k_rem;
    ws.sel[h] = st;
  }
  ghist[255 - tid] = 0u;                                   // clear for the next pass / call
  if (tid == 0) ws.sel_cnt[h] = 0u;
}

struct KeepRule {
  int64_t L, mid_lo, mid_hi;
  uint32_t tau;
  bool none;   // k_mid == 0: keep no middle token
  __device__ __forceinline__ bool protected_pos(int64_t j) const { return j < mid_lo || j >= mid_hi; }
  __device__ __forceinline__ bool above(uint32_t u) const { return !none && u > tau; }
  __device__ __forceinline__ bool tie(uint32_t u) const { return !none && u == tau; }
};

__device__ __forceinline__ KeepRule keep_rule(const HeadTable& ht, const SelState& s, int h) {
  KeepRule r;
  r.L = ht.L;
  r.mid_lo = ht.n_sink;
  r.mid_hi = ht.L - ht.n_recent;
  r.tau = s.tau;
  r.none = ht.k_mid[h] == 0;
  return r;
}

// Per chunk of the whole row: kept tokens that are not ties, and middle ties at tau.
__global__ void __launch_bounds__(kSelThreads)
sel_count_kernel(const float* __restrict__ scores, HeadTable ht, Ws ws, int nchunks,
                 int32_t* __restrict__ cu_out) {
  const int h = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
  if (c == 0 && tid == 0) {
    cu_out[h] = ht.cu[h];
    if (h == ht.Hkv - 1) cu_out[h + 1] = ht.cu[h + 1];
  }
  const KeepRule kr = keep_rule(ht, ws.sel[h], h);
  const int64_t beg = int64_t(c) * kSelChunk;
  const int64_t end = beg + kSelChunk < kr.L ? beg + kSelChunk : kr.L;
  const float* row = scores + int64_t(h) * kr.L;
  uint32_t nk = 0, nt = 0;
  for (int64_t j = beg + tid; j < end; j += blockDim.x) {
    if (kr.protected_pos(j)) {
      ++nk;
      continue;
    }
    const uint32_t u = __float_as_uint(__ldg(row + j));
    nk += kr.above(u);
    nt += kr.tie(u);
  }
  __shared__ uint32_t s_warp[kSelThreads / 32 + 1];
  uint32_t tot_k, tot_t;
  block_excl_scan(nk, s_warp, &tot_k);
  block_excl_scan(nt, s_warp, &tot_t);
  if (tid == 0) ws.chunk_cnt[int64_t(h) * nchunks + c] = make_uint2(tot_k, tot_t);
}

// Writes the kept positions of one chunk at their final place in indices_out.
__global__ void __launch_bounds__(kSelThreads)
sel_write_kernel(const float* __restrict__ scores, HeadTable ht, Ws ws, int nchunks,
                 int32_t* __restrict__ indices_out) {
  const int h = blockIdx.y, c = blockIdx.x, tid = threadIdx.x;
  const SelState st = ws.sel[h];
  const KeepRule kr = keep_rule(ht, st, h);
  __shared__ uint32_t s_warp[kSelThreads / 32 + 1];
  // Totals of the chunks before this one.
  uint32_t bk = 0, bt = 0;
  for (int i = tid; i < c; i += blockDim.x) {
    const uint2 v = ws.chunk_cnt[int64_t(h) * nchunks + i];
    bk += v.x;
    bt += v.y;
  }
  uint32_t before_k, before_t;
  block_excl_scan(bk, s_warp, &before_k);
  block_excl_scan(bt, s_warp, &before_t);
  const uint32_t quota = st.tie_quota;
  const uint32_t ties_left = before_t < quota ? quota - before_t : 0u;
  const uint32_t out_base = uint32_t(ht.cu[h]) + before_k + (before_t < quota ? before_t : quota);

  const int64_t beg = int64_t(c) * kSelChunk + int64_t(tid) * kSelPerThread;
  const float* row = scores + int64_t(h) * kr.L;
  uint32_t u[kSelPerThread];
  uint32_t my_ties = 0;
#pragma unroll
  for (int i = 0; i < kSelPerThread; ++i) {
    const int64_t j = beg + i;
    u[i] = (j < kr.L && !kr.protected_pos(j)) ? __float_as_uint(__ldg(row + j)) : 0u;
    my_ties += (j < kr.L && !kr.protected_pos(j) && kr.tie(u[i])) ? 1u : 0u;
  }
  uint32_t dummy;
  uint32_t tie_rank = block_excl_scan(my_ties, s_warp, &dummy);
  uint32_t keep_mask = 0, my_keep = 0;
#pragma unroll
  for (int i = 0; i < kSelPerThread; ++i) {
    const int64_t j = beg + i;
    bool keep = false;
    if (j < kr.L) {
      if (kr.protected_pos(j)) {
        keep = true;
      } else if (kr.above(u[i])) {
        keep = true;
      } else if (kr.tie(u[i])) {
        keep = tie_rank < ties_left;
        ++tie_rank;
      }
    }
    keep_mask |= uint32_t(keep) << i;
    my_keep += keep;
  }
  uint32_t pos = block_excl_scan(my_keep, s_warp, &dummy) + out_base;
  const uint32_t pos_end = uint32_t(ht.cu[h + 1]);
#pragma unroll
  for (int i = 0; i < kSelPerThread; ++i) {
    if (!(keep_mask & (1u << i))) continue;
    if (pos < pos_end) indices_out[pos] = int32_t(beg + i);
    else record_error(ws.status, SGDKV_ERR_INTERNAL);
    ++pos;
  }
}

// Copies kept rows: 16 threads per 256-byte row of K and of V.
__global__ void __launch_bounds__(256)
gather_kernel(const uint4* __restrict__ K, const uint4* __restrict__ V,
              const int32_t* __restrict__ idx, uint4* __restrict__ Ko, uint4* __restrict__ Vo,
              HeadTable ht, int64_t total_rows, uint32_t* status) {
  const int64_t stride = int64_t(gridDim.x) * blockDim.x;
  for (int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; t < total_rows * 16;
       t += stride) {
    const int64_t o = t >> 4;
    const int part = int(t & 15);
    int lo = 0, hi = ht.Hkv;   // head h with cu[h] <= o < cu[h+1]
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (int64_t(ht.cu[mid]) <= o) lo = mid; else hi = mid;
    }
    const int32_t j = __ldg(idx + o);
    if (j < 0 || int64_t(j) >= ht.L) {
      record_error(status, SGDKV_ERR_INTERNAL);
      continue;
    }
    const int64_t src = (int64_t(lo) * ht.L + j) * 16 + part;
    const uint4 kv = __ldg(K + src);
    const uint4 vv = __ldg(V + src);
    Ko[o * 16 + part] = kv;
    Vo[o * 16 + part] = vv;
  }
}

}  // namespace

cudaError_t launch_compact(const __nv_bfloat16* K, const __nv_bfloat16* V,
                           const float* scores, const HeadTable& ht, int32_t* indices_out,
                           int32_t* cu_out, __nv_bfloat16* K_out, __nv_bfloat16* V_out,
                           int64_t total_rows, const Ws& ws, cudaStream_t stream) {
  const int Hkv = ht.Hkv;
  const int64_t mid = ht.L - ht.n_sink - ht.n_recent;
  const int mid_chunks = int(ceil_div(mid > 0 ? mid : 1, kSelChunk));
  for (int pass = 0; pass < 4; ++pass)
    sel_radix_kernel<<<dim3(mid_chunks, Hkv), kSelThreads, 0, stream>>>(scores, ht, ws, pass,
                                                                         mid_chunks);
  const int row_chunks = int(ceil_div(ht.L, kSelChunk));
  sel_count_kernel<<<dim3(row_chunks, Hkv), kSelThreads, 0, stream>>>(scores, ht, ws,
                                                                      row_chunks, cu_out);
  sel_write_kernel<<<dim3(row_chunks, Hkv), kSelThreads, 0, stream>>>(scores, ht, ws,
                                                                      row_chunks, indices_out);
  note_launches(6);
  if (total_rows > 0) {
    note_launches(1);
    int64_t blocks = ceil_div(total_rows * 16, 256);
    if (blocks > 152 * 16) blocks = 152 * 16;
    gather_kernel<<<int(blocks), 256, 0, stream>>>(
        reinterpret_cast<const uint4*>(K), reinterpret_cast<const uint4*>(V), indices_out,
        reinterpret_cast<uint4*>(K_out), reinterpret_cast<uint4*>(V_out), ht, total_rows,
        ws.status);
  }
  return cudaGetLastError();
}

}  // namespace sgdkv
