// Token selection, ordered compaction and K/V gather (Section 3.3: keep sink and recent
// tokens, then each head's top (b_h - n_sink - n_recent) middle tokens by score; equal
// scores are broken by the lower position).
//
// Scores are finite and non-negative (-0.0 is read as +0.0), so their fp32 bit patterns
// sort like their values and the threshold search is an exact most-significant-digit radix select on uint32 keys:
// four passes of 8-bit digits, each a histogram over the middle keys that match the digits
// fixed so far.  One thread-block cluster works on one KV head: every CTA owns a
// contiguous slice of the row, builds its histogram in shared memory, and after a cluster
// barrier every CTA sums the cluster's histograms (pushed into its shared memory by its
// peers through distributed shared memory) and picks the same digit.  The threshold tau and the number of keys equal to tau to keep
// (lowest positions first) follow.  The same kernel then counts kept positions per slice,
// exchanges the counts through distributed shared memory, and writes every slice's kept
// positions, ascending, at their final offsets.  The kept K/V rows are copied by the
// selection kernel itself when its CTAs span at least kCopyMinCtas SMs (each CTA copies its
// slice's rows), else by a second kernel.
// With a pool source the selection kernel first forms its slice's pooled scores itself
// (the four raw planes summed, then the window maximum, Section 3.3), so the max-pool needs
// no launch of its own.
#include <cooperative_groups.h>

#include <mutex>

#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace cg = cooperative_groups;
namespace {

constexpr int kCThreads = 1024;                // threads per selection CTA
constexpr int kCWarps = kCThreads / 32;
constexpr int kPer = 8;                        // positions per thread per write round
constexpr int kRound = kCThreads * kPer;       // positions per write round

constexpr int kMaxCluster = 16;
static_assert(64 * kMaxCluster <= kCThreads, "one 16-byte histogram piece per thread");
static_assert(32 * kCThreads < 65536, "packed 16-bit slice counts");

// Cross-CTA data is pushed: every CTA stores its histogram (and later its counts) into
// each peer's shared memory, so after the cluster barrier all sums read local memory.
struct SelShared {
  uint32_t wh[kCWarps][256];              // per-warp histograms (neighbouring keys share bins)
  uint32_t hall[2][kMaxCluster][256];     // histograms of every CTA of the cluster, by rank
  __align__(16) uint32_t hsum[256];       // this CTA's histogram of the pass
  uint32_t call[kMaxCluster][2];          // (kept non-ties, ties) of every CTA, by rank
  uint32_t s_warp[kCWarps + 1];
  uint32_t bcast[2];
};

__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

// Exclusive scan of one value per thread over the CTA; *total gets the CTA sum.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* s_warp,
                                                    uint32_t* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  if (lane == 31) s_warp[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    const uint32_t x = lane < kCWarps ? s_warp[lane] : 0u;
    const uint32_t xi = warp_incl_scan(x);
    if (lane < kCWarps) s_warp[lane] = xi - x;
    if (lane == kCWarps - 1) s_warp[kCWarps] = xi;
  }
  __syncthreads();
  const uint32_t r = s_warp[wid] + incl - v;
  *total = s_warp[kCWarps];
  __syncthreads();
  return r;
}

struct KeepRule {
  int64_t mid_lo, mid_hi;
  uint32_t tau;
  bool none;   // nothing selected from the middle
  __device__ __forceinline__ bool protected_pos(int64_t j) const { return j < mid_lo || j >= mid_hi; }
  __device__ __forceinline__ bool above(uint32_t u) const { return !none && u > tau; }
  __device__ __forceinline__ bool tie(uint32_t u) const { return !none && u == tau; }
};

// Radix key of a score: its fp32 bit pattern, with -0.0 read as +0.0 (the two compare
// equal, and the sign bit would otherwise rank -0.0 above every positive score).
__device__ __forceinline__ uint32_t score_key(float s) {
  const uint32_t u = __float_as_uint(s);
  return u == 0x80000000u ? 0u : u;
}

// Shared-memory index of the pool buffer: one word of skew per 32, so that the 16 or so
// consecutive words each thread reads fall into different banks across a warp.
__device__ __forceinline__ int pool_sk(int x) { return x + (x >> 5); }
constexpr int kPoolSmallR = 3;   // window radii up to this take the register path

// The pooled scores of positions p0 .. p0+PER-1 (those inside [beg, end)) as uint32 keys:
// the CTA sums the four planes of its slice and a halo of `radius` positions on each side
// into shared memory (-inf outside the row), then every thread takes the maximum over the
// window [j - radius, j + radius] of each of its positions, in the same arithmetic as the
// stand-alone max-pool kernel, and writes its pooled scores to ps.out.
template <int PER>
__device__ __forceinline__ void pool_slice(const PoolSrc& ps, int h, int64_t L, int64_t beg,
                                           int64_t end, int64_t p0, uint32_t (&u)[PER]) {
  extern __shared__ int32_t stage[];
  float* sum = reinterpret_cast<float*>(stage);       // sum[pool_sk(x)]: position beg - r + x
  const int r = ps.radius;
  const int n = int(end - beg);
  const float* r0 = ps.raw + int64_t(h) * L;
  const int64_t pl = ps.plane;
  const bool cmax = ps.combine_max != 0;
  auto comb = [&](float a, float b, float c, float d) {
    return cmax ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
  };
  auto at = [&](int64_t j) {
    return j >= 0 && j < L ? comb(__ldcg(r0 + j), __ldcg(r0 + pl + j), __ldcg(r0 + 2 * pl + j),
                                  __ldcg(r0 + 3 * pl + j))
                           : -INFINITY;
  };
  const bool vec = ((L | beg | pl) & 3) == 0 && (reinterpret_cast<uintptr_t>(ps.raw) & 15) == 0;
  if (vec) {
    // Rounds of two 16-byte loads per plane and thread, all issued before the first is
    // used; the first round also fetches one position of the halos or of the slice's last
    // n % 4 (at most 2 * kMaxPoolRadius + 3 of them, one per thread).
    const int n4 = n >> 2, nh = 2 * r + (n & 3);
    for (int i0 = threadIdx.x, first = 1; first || i0 < n4; i0 += 2 * kCThreads, first = 0) {
      float4 a[2], b[2], c[2], d[2];
      float hv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      int hx = -1;
      if (first && threadIdx.x < nh) {
        hx = threadIdx.x < r ? threadIdx.x : r + 4 * n4 + (threadIdx.x - r);
        const int64_t j = beg - r + hx;
        if (j >= 0 && j < L) {
#pragma unroll
          for (int k = 0; k < 4; ++k) hv[k] = __ldcg(r0 + k * pl + j);
        }
      }
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int i = i0 + k * kCThreads;
        if (i >= n4) continue;
        const int64_t j = beg + 4 * i;
        a[k] = __ldcg(reinterpret_cast<const float4*>(r0 + j));
        b[k] = __ldcg(reinterpret_cast<const float4*>(r0 + pl + j));
        c[k] = __ldcg(reinterpret_cast<const float4*>(r0 + 2 * pl + j));
        d[k] = __ldcg(reinterpret_cast<const float4*>(r0 + 3 * pl + j));
      }
      if (hx >= 0) sum[pool_sk(hx)] = comb(hv[0], hv[1], hv[2], hv[3]);
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int i = i0 + k * kCThreads;
        if (i >= n4) continue;
        const int x = r + 4 * i;
        sum[pool_sk(x)] = comb(a[k].x, b[k].x, c[k].x, d[k].x);
        sum[pool_sk(x + 1)] = comb(a[k].y, b[k].y, c[k].y, d[k].y);
        sum[pool_sk(x + 2)] = comb(a[k].z, b[k].z, c[k].z, d[k].z);
        sum[pool_sk(x + 3)] = comb(a[k].w, b[k].w, c[k].w, d[k].w);
      }
    }
  } else {
    for (int x = threadIdx.x; x < n + 2 * r; x += kCThreads) sum[pool_sk(x)] = at(beg - r + x);
  }
  __syncthreads();
  const int xb = int(p0 - beg);      // window of position p0 + i: x in [xb + i, xb + i + 2r]
  const int nv = p0 < end ? int(end - p0 < PER ? end - p0 : PER) : 0;   // positions held
  const int lim = nv > 0 ? nv + 2 * r : 0;   // x = xb + k stays below n + 2r
  float m[PER];
  if (r <= kPoolSmallR) {
    float w[PER + 2 * kPoolSmallR];
#pragma unroll
    for (int k = 0; k < PER + 2 * kPoolSmallR; ++k)
      w[k] = k < lim ? sum[pool_sk(xb + k)] : -INFINITY;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      float v = w[i];
#pragma unroll
      for (int k = 1; k <= 2 * kPoolSmallR; ++k)
        if (k <= 2 * r) v = fmaxf(v, w[i + k]);
      m[i] = v;
    }
  } else {
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      float v = -INFINITY;
      if (i < nv)
        for (int k = 0; k <= 2 * r; ++k) v = fmaxf(v, sum[pool_sk(xb + i + k)]);
      m[i] = v;
    }
  }
#pragma unroll
  for (int i = 0; i < PER; ++i) u[i] = i < nv ? score_key(m[i]) : 0u;
  float* o = ps.out + int64_t(h) * L + p0;
  if (nv == PER && PER % 4 == 0 && (reinterpret_cast<uintptr_t>(o) & 15) == 0) {
#pragma unroll
    for (int i = 0; i < PER; i += 4)
      *reinterpret_cast<float4*>(o + i) = make_float4(m[i], m[i + 1], m[i + 2], m[i + 3]);
  } else {
#pragma unroll
    for (int i = 0; i < PER; ++i)
      if (i < nv) o[i] = m[i];
  }
}

// K/V rows to copy from inside the selection kernel (K == nullptr: none; the gather kernel
// copies them instead).
struct RowCopy {
  const uint4* K;
  const uint4* V;
  uint4* Ko;
  uint4* Vo;
};

// One cluster per KV head (grid = Hkv * csize, cluster = csize CTAs).  Control flow is
// uniform across a cluster, so every CTA reaches every cluster barrier.
// PER > 0: each thread holds PER consecutive positions of its CTA's slice in registers for
// the whole kernel (slice <= kCThreads * PER); PER == 0: every pass streams the slice.
// POOL (PER > 0 only): the slice's scores are pooled from ps's raw planes (pool_slice) and
// `scores` is not read.
template <int PER, bool POOL>
__global__ void __launch_bounds__(kCThreads)
sel_cluster_kernel(const float* __restrict__ scores, HeadTable ht, int csize,
                   int32_t* __restrict__ indices_out, int32_t* __restrict__ cu_out,
                   uint32_t* __restrict__ status, PoolSrc ps, RowCopy rc) {
  static_assert(!POOL || PER > 0, "inline pooling needs register-resident slices");
  cg::cluster_group cluster = cg::this_cluster();
  __shared__ SelShared sm;
  const int tid = threadIdx.x, wid = tid >> 5;
  const int rank = int(cluster.block_rank());
  const int h = blockIdx.x / csize;
  const int64_t L = ht.L;
  const int64_t slice = ceil_div(L, csize);
  const int64_t beg = int64_t(rank) * slice < L ? int64_t(rank) * slice : L;
  const int64_t end = beg + slice < L ? beg + slice : L;
  const float* row = scores + int64_t(h) * L;
  KeepRule kr;
  kr.mid_lo = ht.n_sink;
  kr.mid_hi = L - ht.n_recent;
  kr.none = ht.k_mid[h] == 0;
  const int64_t mb = beg > kr.mid_lo ? beg : kr.mid_lo;     // middle part of this slice
  const int64_t me = end < kr.mid_hi ? end : kr.mid_hi;

  // register-resident positions p0 .. p0+PER-1 (0 bits outside the slice: never read)
  const int64_t p0 = beg + int64_t(tid) * (PER > 0 ? PER : 1);
  uint32_t u[PER > 0 ? PER : 1];
  // The first push into a peer's shared memory may only happen once every CTA of the
  // cluster runs: arrive here, wait after the slice is loaded (long since complete by then).
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  if constexpr (POOL) {
    pool_slice<PER>(ps, h, L, beg, end, p0, u);
  } else if constexpr (PER > 0) {
#pragma unroll
    for (int i = 0; i < PER; ++i) u[i] = p0 + i < end ? score_key(__ldg(row + p0 + i)) : 0u;
  }

  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");

  uint32_t cand = 0u;                       // PER > 0: bit i = position p0+i is middle
  if constexpr (PER > 0) {
#pragma unroll
    for (int i = 0; i < PER; ++i)
      if (p0 + i >= mb && p0 + i < me) cand |= 1u << i;
  }

  // ---- radix select of tau over the middle of the row --------------------------------
  uint32_t prefix = 0u, k_rem = uint32_t(ht.k_mid[h]);
  if (!kr.none) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      const uint32_t hi_mask = pass == 0 ? 0u : (0xffffffffu << (32 - 8 * pass));
      for (int i = tid & 31; i < 256; i += 32) sm.wh[wid][i] = 0u;
      __syncwarp();
      if constexpr (PER > 0) {
        // cand: this thread's middle positions still matching the digits fixed so far.
        // Lanes of a warp that hit the same bin add once (neighbouring positions have
        // similar scores, so a warp's keys fall into few bins).
        // A thread's positions are consecutive and pooled scores come in runs, so equal
        // digits are counted in a register and added once per run.
        uint32_t keep = 0u, run_bin = 0u, run_len = 0u;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
          const bool take = ((cand >> i) & 1u) && (u[i] & hi_mask) == prefix;
          keep |= uint32_t(take) << i;
          if (take) {
            const uint32_t d = (u[i] >> shift) & 255u;
            if (run_len && d != run_bin) {
              atomicAdd(&sm.wh[wid][run_bin], run_len);
              run_len = 0u;
            }
            run_bin = d;
            ++run_len;
          }
        }
        if (run_len) atomicAdd(&sm.wh[wid][run_bin], run_len);
        cand = keep;
      } else {
#pragma unroll 4
        for (int64_t j = mb + tid; j < me; j += kCThreads) {
          const uint32_t x = score_key(__ldg(row + j));
          if ((x & hi_mask) == prefix) atomicAdd(&sm.wh[wid][(x >> shift) & 255u], 1u);
        }
      }
      __syncthreads();
      if (tid < 256) {
        uint32_t c = 0;
#pragma unroll
        for (int w = 0; w < kCWarps; ++w) c += sm.wh[w][tid];
        sm.hsum[tid] = c;
      }
      __syncthreads();
      if (tid < 64 * csize) {               // push: one 16-byte quarter-row to one peer each
        const int r = tid >> 6, qd = tid & 63;
        const uint4 v = reinterpret_cast<const uint4*>(sm.hsum)[qd];
        reinterpret_cast<uint4*>(cluster.map_shared_rank(&sm.hall[pass & 1][rank][0], r))[qd] = v;
      }
      cluster.sync();                       // every slice's histogram has arrived
      // thread t < 256 takes bin 255 - t: descending digit order
      uint32_t cnt = 0;
      if (tid < 256)
        for (int r = 0; r < csize; ++r) cnt += sm.hall[pass & 1][r][255 - tid];
      uint32_t total;
      const uint32_t excl = block_excl_scan(cnt, sm.s_warp, &total);
      if (tid < 256 && excl < k_rem && excl + cnt >= k_rem) {   // exactly one thread
        sm.bcast[0] = prefix | (uint32_t(255 - tid) << shift);
        sm.bcast[1] = k_rem - excl;
      }
      __syncthreads();
      prefix = sm.bcast[0];
      k_rem = sm.bcast[1];
      // hall[pass & 1] is rewritten two passes later, after the next cluster barrier,
      // which every CTA reaches only once it has finished reading it.
    }
  }
  kr.tau = prefix;
  const uint32_t quota = kr.none ? 0u : k_rem;            // keys equal to tau to keep

  // ---- kept positions per slice, exchanged across the cluster --------------------------
  uint32_t nk = 0, nt = 0;
  if constexpr (PER > 0) {
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int64_t j = p0 + i;
      if (j >= end) continue;
      if (kr.protected_pos(j)) {
        ++nk;
        continue;
      }
      nk += kr.above(u[i]);
      nt += kr.tie(u[i]);
    }
  } else {
    for (int64_t j = beg + tid; j < end; j += kCThreads) {
      if (kr.protected_pos(j)) {
        ++nk;
        continue;
      }
      const uint32_t x = score_key(__ldg(row + j));
      nk += kr.above(x);
      nt += kr.tie(x);
    }
  }
  uint32_t tot_k, tot_t, my_k_before, my_t_before;
  if constexpr (PER > 0) {
    // both counts in one scan: a CTA holds at most 32 * 1024 positions, below 2^16
    uint32_t tot;
    const uint32_t before = block_excl_scan((nk << 16) | nt, sm.s_warp, &tot);
    my_k_before = before >> 16;
    my_t_before = before & 0xffffu;
    tot_k = tot >> 16;
    tot_t = tot & 0xffffu;
  } else {
    my_k_before = block_excl_scan(nk, sm.s_warp, &tot_k);
    my_t_before = block_excl_scan(nt, sm.s_warp, &tot_t);
  }
  if (tid < csize) {                        // push this slice's counts to CTA `tid`
    uint32_t* dst = cluster.map_shared_rank(&sm.call[rank][0], tid);
    dst[0] = tot_k;
    dst[1] = tot_t;
  }
  cluster.sync();
  if (tid == 0) {
    uint32_t bk = 0, bt = 0;
    for (int r = 0; r < rank; ++r) {
      bk += sm.call[r][0];
      bt += sm.call[r][1];
    }
    sm.bcast[0] = bk;
    sm.bcast[1] = bt;
  }
  __syncthreads();
  const uint32_t before_k = sm.bcast[0], before_t = sm.bcast[1];
  uint32_t ties_left = before_t < quota ? quota - before_t : 0u;
  uint32_t out = uint32_t(ht.cu[h]) + before_k + (before_t < quota ? before_t : quota);
  const uint32_t out_end = uint32_t(ht.cu[h + 1]);

  if constexpr (PER > 0) {
    // ---- ordered write from registers (thread order = position order), staged in shared
    // memory so the copy to indices_out is coalesced ---------------------------------------
    extern __shared__ int32_t stage[];                  // kCThreads * PER kept positions
    uint32_t tie_rank = my_t_before;
    uint32_t slot = my_k_before + (my_t_before < ties_left ? my_t_before : ties_left);
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int64_t j = p0 + i;
      if (j >= end) continue;
      bool keep;
      if (kr.protected_pos(j)) {
        keep = true;
      } else if (kr.above(u[i])) {
        keep = true;
      } else if (kr.tie(u[i])) {
        keep = tie_rank < ties_left;
        ++tie_rank;
      } else {
        keep = false;
      }
      if (!keep) continue;
      if (slot < uint32_t(kCThreads * PER)) stage[slot] = int32_t(j);
      else record_error(status, SGDKV_ERR_INTERNAL);
      ++slot;
    }
    __syncthreads();
    const uint32_t kept = tot_k + (tot_t < ties_left ? tot_t : ties_left);
    for (uint32_t i = tid; i < kept && i < uint32_t(kCThreads * PER); i += kCThreads) {
      if (out + i < out_end) indices_out[out + i] = stage[i];
      else record_error(status, SGDKV_ERR_INTERNAL);
    }
    if (rc.K) {
      // ---- the slice's kept K and V rows, copied here (16 threads per 256-byte row, two
      // rows per thread in flight; read and written once: streaming loads and stores)
      constexpr uint32_t kRowsPerPass = kCThreads / 16;
      const int part = tid & 15;
      const int64_t hrow = int64_t(h) * L;
      const uint32_t nk = kept < uint32_t(kCThreads * PER) ? kept : uint32_t(kCThreads * PER);
      for (uint32_t i0 = uint32_t(tid >> 4); i0 < nk; i0 += 2 * kRowsPerPass) {
        const uint32_t i1 = i0 + kRowsPerPass;
        const bool ok0 = out + i0 < out_end, ok1 = i1 < nk && out + i1 < out_end;
        uint4 k0, v0, k1, v1;
        if (ok0) {
          const int64_t src = (hrow + stage[i0]) * 16 + part;
          k0 = __ldcs(rc.K + src);
          v0 = __ldcs(rc.V + src);
        }
        if (ok1) {
          const int64_t src = (hrow + stage[i1]) * 16 + part;
          k1 = __ldcs(rc.K + src);
          v1 = __ldcs(rc.V + src);
        }
        if (ok0) {
          __stcs(rc.Ko + int64_t(out + i0) * 16 + part, k0);
          __stcs(rc.Vo + int64_t(out + i0) * 16 + part, v0);
        }
        if (ok1) {
          __stcs(rc.Ko + int64_t(out + i1) * 16 + part, k1);
          __stcs(rc.Vo + int64_t(out + i1) * 16 + part, v1);
        }
      }
    }
  } else {
    // ---- ordered write, rounds of kRound positions -------------------------------------
    for (int64_t r0 = beg; r0 < end; r0 += kRound) {
      const int64_t q0 = r0 + int64_t(tid) * kPer;
      uint32_t x[kPer];
      uint32_t my_ties = 0;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const int64_t j = q0 + i;
        const bool mid = j < end && !kr.protected_pos(j);
        x[i] = mid ? score_key(__ldg(row + j)) : 0u;
        my_ties += (mid && kr.tie(x[i])) ? 1u : 0u;
      }
      uint32_t round_ties;
      uint32_t tie_rank = block_excl_scan(my_ties, sm.s_warp, &round_ties);
      uint32_t keep_mask = 0, my_keep = 0;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        const int64_t j = q0 + i;
        bool keep = false;
        if (j < end) {
          if (kr.protected_pos(j)) {
            keep = true;
          } else if (kr.above(x[i])) {
            keep = true;
          } else if (kr.tie(x[i])) {
            keep = tie_rank < ties_left;
            ++tie_rank;
          }
        }
        keep_mask |= uint32_t(keep) << i;
        my_keep += keep;
      }
      uint32_t round_kept;
      uint32_t pos = block_excl_scan(my_keep, sm.s_warp, &round_kept) + out;
#pragma unroll
      for (int i = 0; i < kPer; ++i) {
        if (!(keep_mask & (1u << i))) continue;
        if (pos < out_end) indices_out[pos] = int32_t(q0 + i);
        else record_error(status, SGDKV_ERR_INTERNAL);
        ++pos;
      }
      out += round_kept;
      ties_left = round_ties < ties_left ? ties_left - round_ties : 0u;
    }
  }
  if (rank == 0 && tid == 0) {
    cu_out[h] = ht.cu[h];
    if (h == ht.Hkv - 1) cu_out[h + 1] = ht.cu[h + 1];
  }
  // No barrier before leaving: the last stores into a peer's shared memory (the kept
  // counts) precede the cluster barrier above, so no peer touches this CTA's shared memory
  // any more.
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
    // rows read and written once: streaming (evict-first) loads and stores, so that the copy
    // does not push out of L2 the key tiles pass 2 of the next layer is about to re-read
    const uint4 kv = __ldcs(K + src);
    const uint4 vv = __ldcs(V + src);
    __stcs(Ko + o * 16 + part, kv);
    __stcs(Vo + o * 16 + part, vv);
  }
}

// Dynamic shared memory of a selection kernel: the staged kept positions, and with POOL
// the pool buffer of a slice and its halos (skewed), which it precedes.
template <int PER, bool POOL>
constexpr size_t sel_smem_bytes() {
  const size_t st = size_t(kCThreads) * (PER > 0 ? PER : 0) * sizeof(int32_t);
  const size_t pb = POOL ? size_t(kCThreads * PER + 2 * kMaxPoolRadius) * 33 / 32 + 1 : 0;
  return st > pb * sizeof(float) ? st : pb * sizeof(float);
}

// Largest cluster size (16 if the device runs it, else the portable 8) for the selection.
// The kernel's shared-memory and cluster-size attributes belong to the device that is
// current when they are set, so they are set, and the size found, once per device, under a
// lock (host threads may launch on several devices at once).
constexpr int kMaxSelDevices = 64;

template <int PER, bool POOL>
int probe_cluster_size() {
  int size = 8;
  constexpr size_t smem = sel_smem_bytes<PER, POOL>();
  cudaFuncSetAttribute(sel_cluster_kernel<PER, POOL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       int(smem));
  if (cudaFuncSetAttribute(sel_cluster_kernel<PER, POOL>,
                           cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(16, 1, 1);
    cfg.blockDim = dim3(kCThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 16;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxPotentialClusterSize(&n, sel_cluster_kernel<PER, POOL>, &cfg) ==
            cudaSuccess &&
        n >= 16)
      size = 16;
  }
  cudaGetLastError();   // a refused query leaves the portable size
  return size;
}

template <int PER, bool POOL>
int cluster_size() {
  static std::mutex mu;
  static int cached[kMaxSelDevices] = {};
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxSelDevices) {
    cudaGetLastError();
    return probe_cluster_size<PER, POOL>();      // no slot to cache in: set up every call
  }
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev] == 0) cached[dev] = probe_cluster_size<PER, POOL>();
  return cached[dev];
}

template <int PER, bool POOL>
cudaError_t launch_select(const float* scores, const HeadTable& ht, int csize,
                          int32_t* indices_out, int32_t* cu_out, uint32_t* status,
                          const PoolSrc& ps, const RowCopy& rc, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(ht.Hkv * csize), 1, 1);
  cfg.blockDim = dim3(kCThreads, 1, 1);
  cfg.dynamicSmemBytes = sel_smem_bytes<PER, POOL>();
  cfg.stream = stream;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = unsigned(csize);
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sel_cluster_kernel<PER, POOL>, scores, ht, csize,
                            indices_out, cu_out, status, ps, rc);
}

// Positions per thread of the selection kernel for rows of length L: slices of up to 32
// positions per thread stay in registers for the whole kernel (the positions per thread
// follow from the cluster size that kernel actually runs with); 0: the streaming kernel.
// Rows short enough for 8 positions per thread on fewer CTAs are selected by clusters of
// this many CTAs or more (measured on the benchmark's step, 32K rows and 4 KV heads: 16-CTA
// clusters 783 M, 8-CTA 830 M, 4-CTA 825 M tokens/s/layer; 4K rows: 1-CTA clusters 66 M
// against 79-80 M).
constexpr int kMinShortCluster = 8;

template <bool POOL>
int pick_per(int64_t L, int* csize) {
  auto fits = [&](int per, int cs) { return ceil_div(ceil_div(L, cs), kCThreads) <= per; };
  if (fits(8, *csize = cluster_size<8, POOL>())) {
    // short rows: the smallest cluster of at least kMinShortCluster CTAs whose slices still
    // fit (fewer peers to push histograms to, and SMs left to the scoring kernels)
    while (*csize > kMinShortCluster && fits(8, *csize - 1)) --*csize;
    return 8;
  }
  if (fits(16, *csize = cluster_size<16, POOL>())) return 16;
  if (fits(32, *csize = cluster_size<32, POOL>())) return 32;
  *csize = cluster_size<0, false>();
  return 0;
}

// The selection copies the kept K/V rows itself when its CTAs span at least this many SMs:
// each CTA moves its slice's rows with ordinary loads and stores, so on fewer SMs the copy
// is slower than the gather kernel's, which spreads over the whole GPU (measured on the
// benchmark's two-stream step: 4 KV heads, 64 CTAs, 1.2 % slower; 8 KV heads, 128 CTAs,
// 4.7 % faster).
constexpr int kCopyMinCtas = 128;

// rc: the rows to copy when the selection keeps its slices in registers and spans at least
// kCopyMinCtas CTAs (then *copied is set); otherwise the gather kernel copies them.
template <bool POOL>
cudaError_t dispatch_select(const float* scores, const HeadTable& ht, int32_t* indices_out,
                            int32_t* cu_out, uint32_t* status, const PoolSrc& ps,
                            const RowCopy& rc_in, bool* copied, cudaStream_t stream) {
  int cs = 0;
  const int per = pick_per<POOL>(ht.L, &cs);
  *copied = per > 0 && rc_in.K != nullptr && ht.Hkv * cs >= kCopyMinCtas;
  const RowCopy rc = *copied ? rc_in : RowCopy{nullptr, nullptr, nullptr, nullptr};
  switch (per) {
    case 8:
      return launch_select<8, POOL>(scores, ht, cs, indices_out, cu_out, status, ps, rc, stream);
    case 16:
      return launch_select<16, POOL>(scores, ht, cs, indices_out, cu_out, status, ps, rc, stream);
    case 32:
      return launch_select<32, POOL>(scores, ht, cs, indices_out, cu_out, status, ps, rc, stream);
    default:
      if (POOL) return cudaErrorInvalidValue;   // callers check compact_pools_inline
      return launch_select<0, false>(scores, ht, cs, indices_out, cu_out, status, ps,
                                     RowCopy{nullptr, nullptr, nullptr, nullptr}, stream);
  }
}

}  // namespace

cudaError_t launch_compact(const __nv_bfloat16* K, const __nv_bfloat16* V,
                           const float* scores, const HeadTable& ht, int32_t* indices_out,
                           int32_t* cu_out, __nv_bfloat16* K_out, __nv_bfloat16* V_out,
                           int64_t total_rows, const Ws& ws, cudaStream_t stream,
                           const PoolSrc* pool_src) {
  cudaError_t e;
  bool copied = false;
  const RowCopy rc = total_rows > 0
                         ? RowCopy{reinterpret_cast<const uint4*>(K),
                                   reinterpret_cast<const uint4*>(V),
                                   reinterpret_cast<uint4*>(K_out), reinterpret_cast<uint4*>(V_out)}
                         : RowCopy{nullptr, nullptr, nullptr, nullptr};
  {
    KernelTimer t(SGDKV_KERNEL_SELECT, stream);
    if (pool_src)
      e = dispatch_select<true>(pool_src->out, ht, indices_out, cu_out, ws.status, *pool_src, rc,
                                &copied, stream);
    else
      e = dispatch_select<false>(scores, ht, indices_out, cu_out, ws.status, PoolSrc{}, rc,
                                 &copied, stream);
  }
  if (e != cudaSuccess) return e;
  note_launches(1);
  if (total_rows > 0 && !copied) {
    KernelTimer tg(SGDKV_KERNEL_GATHER, stream);
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

bool compact_pools_inline(int64_t L) {
  int cs = 0;
  return pick_per<true>(L, &cs) > 0;
}

}  // namespace sgdkv
