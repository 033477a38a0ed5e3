// Decode attention over the compressed cache (the consumer of the compression step): for
// every query head qh and new token t, out[qh, t] = sum_i softmax_i(q . k_i / sqrt(d)) v_i
// over the kept rows i of KV head qh / G (Section 3.3: the retained tokens are the heads'
// history; Appendix, Configuration: the cache is kept per KV head, before the values are
// repeated for the query heads of a GQA group).  The cache is the flat [sum b_h][d] pair
// that sgdkv_compact writes, head h's rows at [cu[h], cu[h+1]).
//
// The work is a stream of the kept K and V rows (HBM-bound: G * T <= 16 query rows meet
// every K row once and every V row once).  Each warp takes a contiguous chunk of one head's
// rows (a quarter of its CTA's chunk) and streams it through a three-stage ring of 32-row K
// and V tiles in its own shared
// memory (cp.async, 16-byte chunks, XOR-swizzled so that the matrix loads are free of bank
// conflicts).  Per tile, 16 x 32 logits come from mma.m16n8k16 (bf16, fp32 accumulate; the
// query rows of the group are the 16 rows of A, padded with zeros), an online softmax in
// log2 units runs per query row across the four threads that hold it, and the weights,
// rounded to bf16, multiply the V tile in a second mma chain into 16 x 128 fp32
// accumulators.  The row sums are taken over the rounded weights, so every output is a
// convex combination of the head's value rows.  The four warps of a CTA merge their (max,
// sum, 128 sums) per query row in shared memory into one partial per CTA chunk; a second
// kernel merges a head's partials.  Both kernels are programmatic dependents of what
// precedes them: the merge's blocks wait in hardware for the partials, and the partial
// kernel of a call that follows another decode call streams its cache while the previous
// merge runs, writing its partials only after that merge has completed.
#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace {

constexpr int kDWarps = 4;                 // warps per CTA (a quarter of the CTA's chunk each)
constexpr int kDTile = 32;                 // rows per tile
constexpr int kDStages = 3;                // tiles in flight per warp
constexpr int kDTileBytes = kDTile * kD * 2;            // 8 KB of K or of V
constexpr int kDWarpBytes = kDStages * 2 * kDTileBytes;  // 48 KB per warp
constexpr int kDPartStride = kD + 4;       // floats per partial row: 128 sums, max, sum, pad
constexpr int kDTargetChunks = 152;       // CTA chunks per call: one wave on 152 SMs

struct DecodeParams {
  int Hkv, G, T, nq;                       // nq = G * T query rows per head (<= 16)
  int chunk;                               // rows per CTA chunk (a multiple of kDWarps*kDTile)
  float scale2;                            // log2(e) / sqrt(d)
  int32_t cu[SGDKV_MAX_KV_HEADS + 1];      // first row of each head in the flat cache
  int32_t wpfx[SGDKV_MAX_KV_HEADS + 1];    // first CTA chunk of each head
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
// 16 bytes global -> shared, zero-filled beyond src_bytes (0 or 16)
__device__ __forceinline__ void cp16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                          uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// D += A (16 x 16 bf16, row) * B (16 x 8 bf16, col), fp32
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// two floats -> bf16x2 (round to nearest even; the lower index in the low half), and the
// rounded values back
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi, float& rlo, float& rhi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  rlo = __low2float(v);
  rhi = __high2float(v);
  return *reinterpret_cast<const uint32_t*>(&v);
}
// byte offset of 16-byte chunk c of tile row r (chunks XOR-swizzled by the row's low bits)
__device__ __forceinline__ uint32_t tile_off(int r, int c) {
  return uint32_t(r * (kD * 2) + ((c ^ (r & 7)) << 4));
}

__global__ void __launch_bounds__(kDWarps * 32)
decode_partial_kernel(const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ Kc,
                      const __nv_bfloat16* __restrict__ Vc, DecodeParams p,
                      float* __restrict__ part) {
  extern __shared__ __align__(128) uint8_t dsm[];
  // the merge kernel may be scheduled now: its blocks wait for this grid's results
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int cg = blockIdx.x;                             // CTA chunk (grid = chunks)
  int h = 0;
  while (cg >= p.wpfx[h + 1]) ++h;
  const int c0 = p.cu[h] + (cg - p.wpfx[h]) * p.chunk;
  const int c1 = min(c0 + p.chunk, p.cu[h + 1]);
  const int sub = p.chunk / kDWarps;                     // this warp: a quarter of the chunk
  const int row0 = min(c0 + warp * sub, c1);
  const int row_end = min(row0 + sub, c1);
  const int ntiles = (row_end - row0 + kDTile - 1) / kDTile;
  uint8_t* wbase = dsm + warp * kDWarpBytes;
  const uint32_t sbase = smem_addr(wbase);

  // tile i (rows row0 + 32 i ...) into stage i % kDStages: K then V, 16-byte chunks; rows
  // past the chunk are zero-filled
  auto load_tile = [&](int i) {
    const uint32_t kd = sbase + uint32_t((i % kDStages) * 2 * kDTileBytes);
    const uint32_t vd = kd + kDTileBytes;
#pragma unroll
    for (int k = 0; k < (kDTile * 16) / 32; ++k) {
      const int c = lane + 32 * k, r = c >> 4, ch = c & 15;
      const int row = row0 + i * kDTile + r;
      const bool ok = row < row_end;
      const size_t src = size_t(ok ? row : row0) * kD + ch * 8;
      cp16(kd + tile_off(r, ch), Kc + src, ok ? 16u : 0u);
      cp16(vd + tile_off(r, ch), Vc + src, ok ? 16u : 0u);
    }
  };

  // the group's query rows as A fragments, zero past nq (q rows of head h: h * nq ...)
  uint32_t qa[8][4];
  {
    const __nv_bfloat16* qh = q + size_t(h) * p.nq * kD;
    const uint32_t* q0 = reinterpret_cast<const uint32_t*>(qh + size_t(g) * kD);
    const uint32_t* q1 = reinterpret_cast<const uint32_t*>(qh + size_t(g + 8) * kD);
#pragma unroll
    for (int kc = 0; kc < 8; ++kc) {
      qa[kc][0] = g < p.nq ? __ldg(q0 + kc * 8 + t) : 0u;
      qa[kc][1] = g + 8 < p.nq ? __ldg(q1 + kc * 8 + t) : 0u;
      qa[kc][2] = g < p.nq ? __ldg(q0 + kc * 8 + 4 + t) : 0u;
      qa[kc][3] = g + 8 < p.nq ? __ldg(q1 + kc * 8 + 4 + t) : 0u;
    }
  }
  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;   // rows g and g + 8

#pragma unroll
  for (int i = 0; i < kDStages - 1; ++i) {
    if (i < ntiles) load_tile(i);
    cp_commit();
  }
  for (int i = 0; i < ntiles; ++i) {
    if (i + kDStages - 1 < ntiles) load_tile(i + kDStages - 1);
    cp_commit();
    cp_wait<kDStages - 1>();                 // tile i has landed
    __syncwarp();
    const uint32_t kt = sbase + uint32_t((i % kDStages) * 2 * kDTileBytes);
    const uint32_t vt = kt + kDTileBytes;
    // logits: 4 column tiles of 8 rows (keys) x 16 query rows
    float s[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
      for (int kc = 0; kc < 8; kc += 2) {
        uint32_t b0, b1, b2, b3;
        const int r = 8 * j + (lane & 7), ch = 2 * kc + (lane >> 3);
        ldsm_x4(kt + tile_off(r, ch), b0, b1, b2, b3);
        mma16816(s[j], qa[kc], b0, b1);
        mma16816(s[j], qa[kc + 1], b2, b3);
      }
    }
    // rows of this tile past the chunk take no part
    const int valid = row_end - (row0 + i * kDTile);
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const bool ok = 8 * j + 2 * t + e < valid;
        s[j][e] = ok ? s[j][e] * p.scale2 : -INFINITY;
        s[j][2 + e] = ok ? s[j][2 + e] * p.scale2 : -INFINITY;
        mx0 = fmaxf(mx0, s[j][e]);
        mx1 = fmaxf(mx1, s[j][2 + e]);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);    // > -inf: valid >= 1
    const float a0 = m0 == -INFINITY ? 0.f : ex2f(m0 - n0);
    const float a1 = m1 == -INFINITY ? 0.f : ex2f(m1 - n1);
    m0 = n0;
    m1 = n1;
    l0 *= a0;
    l1 *= a1;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= a0;
      o[n][1] *= a0;
      o[n][2] *= a1;
      o[n][3] *= a1;
    }
    // weights (bf16) as A fragments of two 16-row steps, their rounded values summed
    uint32_t pa[2][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float r0, r1, r2, r3;
      const uint32_t lo = pack_bf16(ex2f(s[j][0] - n0), ex2f(s[j][1] - n0), r0, r1);
      const uint32_t hi = pack_bf16(ex2f(s[j][2] - n1), ex2f(s[j][3] - n1), r2, r3);
      l0 += r0 + r1;
      l1 += r2 + r3;
      pa[j >> 1][(j & 1) * 2 + 0] = lo;
      pa[j >> 1][(j & 1) * 2 + 1] = hi;
    }
    // out += weights (16 x 32) * V tile (32 x 128)
#pragma unroll
    for (int ks = 0; ks < 2; ++ks) {
#pragma unroll
      for (int n = 0; n < 16; n += 2) {
        uint32_t b0, b1, b2, b3;
        const int mi = lane >> 3;
        const int r = 16 * ks + 8 * (mi & 1) + (lane & 7), ch = n + (mi >> 1);
        ldsm_x4_t(vt + tile_off(r, ch), b0, b1, b2, b3);
        mma16816(o[n], pa[ks], b0, b1);
        mma16816(o[n + 1], pa[ks], b2, b3);
      }
    }
    __syncwarp();                              // stage i % kDStages free for refill
  }
  cp_wait<0>();
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  // the four warps' (max, sum, 128 sums) per row, in the rings' shared memory once every
  // warp is done with its ring, merged by one thread per column into the CTA's partial
  __syncthreads();
  float* red = reinterpret_cast<float*>(dsm);            // [kDWarps][16][kDPartStride]
  float* r0 = red + (warp * 16 + g) * kDPartStride;
  float* r1 = red + (warp * 16 + g + 8) * kDPartStride;
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    *reinterpret_cast<float2*>(r0 + 8 * n + 2 * t) = make_float2(o[n][0], o[n][1]);
    *reinterpret_cast<float2*>(r1 + 8 * n + 2 * t) = make_float2(o[n][2], o[n][3]);
  }
  if (t == 0) {
    r0[kD] = m0;
    r0[kD + 1] = l0;
    r1[kD] = m1;
    r1[kD + 1] = l1;
  }
  __syncthreads();
  // launched as a programmatic dependent of the previous call's merge: the streaming above
  // overlapped it, and the partials it reads are rewritten only once it has completed
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int d = threadIdx.x;                             // kDWarps * 32 == kD columns
  for (int r = 0; r < p.nq; ++r) {
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kDWarps; ++w) M = fmaxf(M, red[(w * 16 + r) * kDPartStride + kD]);
    float S = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < kDWarps; ++w) {
      const float* rw = red + (w * 16 + r) * kDPartStride;
      const float f = rw[kD] == -INFINITY ? 0.f : ex2f(rw[kD] - M);
      S += f * rw[kD + 1];
      O += f * rw[d];
    }
    float* pr = part + (size_t(cg) * 16 + r) * kDPartStride;
    pr[d] = O;
    if (d == 0) {
      pr[kD] = M;
      pr[kD + 1] = S;
    }
  }
}

// out[h * nq + r][d] = sum_w 2^(m_w - M) o_w[d] / sum_w 2^(m_w - M) l_w over the head's CTA
// chunks w (zeros for a head without rows).  One block per (head, query row), one global
// round trip: eight groups of 64 threads (one column pair each) take the partials w = g,
// g + 8, ...; with its column pair of up to kDCombU of them a thread loads the (max, sum) of
// one of its group's partials, which reach the group through shared memory (a head has at
// most kDTargetChunks + 1 chunks: one round of loads covers it); each thread folds its
// partials into a running (max, weighted sums), and the block combines the threads' results
// against the block's maximum.
constexpr int kDCombThreads = 512;
constexpr int kDMaxChunks = 1024;              // >= kDTargetChunks + SGDKV_MAX_KV_HEADS
constexpr int kDCombGroups = kDCombThreads / 64;
constexpr int kDCombU = 20;                    // partials per thread and round trip
static_assert(kDCombGroups * kDCombU >= kDTargetChunks + 1, "one round trip per head");

__device__ __forceinline__ float block_reduce(float v, bool is_max, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float x = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, x) : v + x;
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  v = is_max ? -INFINITY : 0.f;
  for (int i = 0; i < kDCombThreads / 32; ++i) v = is_max ? fmaxf(v, red[i]) : v + red[i];
  __syncthreads();
  return v;
}

__global__ void __launch_bounds__(kDCombThreads)
decode_combine_kernel(const float* __restrict__ part, DecodeParams p, float* __restrict__ out) {
  __shared__ float red[kDCombThreads / 32];
  __shared__ float2 osum[kDCombGroups][kD / 2];
  __shared__ float2 sml[kDCombGroups][kDCombU];   // (max, sum) of a group's partials
  const int h = blockIdx.x / p.nq, r = blockIdx.x % p.nq, tid = threadIdx.x;
  const int w0 = p.wpfx[h], n = min(p.wpfx[h + 1] - w0, kDMaxChunks);
  auto row = [&](int w) { return part + (size_t(w0 + w) * 16 + r) * kDPartStride; };
  // the next call's partial kernel may be scheduled now (it writes the partials only after
  // this grid has completed)
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // launched as a programmatic dependent of the partial kernel: the partials are complete
  // and visible once this returns (a no-op after an ordinary launch)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int grp = tid >> 6, cp = tid & 63;       // column pair 2 cp, 2 cp + 1
  float mt = -INFINITY, st = 0.f;                // this thread's running max and sum
  float2 o = make_float2(0.f, 0.f);
  for (int base = 0; base < n; base += kDCombGroups * kDCombU) {
    const int w = base + grp;
    // partial w + 8 k of this group: a fixed stride from partial w (one base address)
    constexpr size_t kStep = size_t(kDCombGroups) * 16 * kDPartStride / 2;   // in float2
    const float2* pv = reinterpret_cast<const float2*>(part) +
                       (size_t(w0 + w) * 16 + r) * (kDPartStride / 2) + cp;
    float2 v[kDCombU];
#pragma unroll
    for (int k = 0; k < kDCombU; ++k)
      v[k] = w + kDCombGroups * k < n ? __ldcg(pv + kStep * k) : make_float2(0.f, 0.f);
    if (cp < kDCombU) {
      const int wk = w + kDCombGroups * cp;
      sml[grp][cp] = wk < n ? __ldcg(reinterpret_cast<const float2*>(row(wk) + kD))
                            : make_float2(-INFINITY, 0.f);
    }
    __syncthreads();
    float mb = mt;
#pragma unroll
    for (int k = 0; k < kDCombU; ++k) mb = fmaxf(mb, sml[grp][k].x);
    if (mb != -INFINITY) {
      const float sc = mt == -INFINITY ? 0.f : ex2f(mt - mb);
      o.x *= sc;
      o.y *= sc;
      st *= sc;
#pragma unroll
      for (int k = 0; k < kDCombU; ++k) {
        const float2 e = sml[grp][k];
        const float fw = e.x == -INFINITY ? 0.f : ex2f(e.x - mb);
        o.x += fw * v[k].x;
        o.y += fw * v[k].y;
        st += fw * e.y;
      }
      mt = mb;
    }
    __syncthreads();                             // sml is rewritten by the next round
  }
  const float M = block_reduce(mt, true, red);
  const float sc = mt == -INFINITY ? 0.f : ex2f(mt - M);
  o.x *= sc;
  o.y *= sc;
  const float S = block_reduce(cp == 0 ? st * sc : 0.f, false, red);   // one sum per group
  osum[grp][cp] = o;
  __syncthreads();
  if (tid < kD / 2) {
    float2 O = make_float2(0.f, 0.f);
#pragma unroll
    for (int g = 0; g < kDCombGroups; ++g) {
      O.x += osum[g][tid].x;
      O.y += osum[g][tid].y;
    }
    const float inv = S > 0.f ? 1.f / S : 0.f;
    *reinterpret_cast<float2*>(out + (size_t(h) * p.nq + r) * kD + 2 * tid) =
        make_float2(O.x * inv, O.y * inv);
  }
}

}  // namespace

// Rows per CTA chunk: about kDTargetChunks chunks per call, a whole tile per warp (a
// function of the total rows alone, so that the workspace size does not depend on the
// device).
int decode_chunk_rows(int64_t total_rows) {
  constexpr int kQuant = kDWarps * kDTile;
  int64_t c = ceil_div(total_rows > 0 ? total_rows : 1, kDTargetChunks);
  c = ceil_div(c, kQuant) * kQuant;
  return int(c);
}

// Bytes of the partials: one per CTA chunk, at most min(ceil(rows / (kDWarps * kDTile)),
// kDTargetChunks) + Hkv of them (a chunk holds >= kDWarps * kDTile and >= rows /
// kDTargetChunks rows).  The bound grows with total_rows, so a workspace sized for the
// largest cache serves every smaller one.
size_t decode_partial_bytes(int64_t total_rows, int Hkv) {
  int64_t n = ceil_div(total_rows, kDWarps * kDTile);
  if (n > kDTargetChunks) n = kDTargetChunks;
  return size_t(n + Hkv) * 16 * kDPartStride * sizeof(float);
}

cudaError_t launch_decode(const __nv_bfloat16* q, const __nv_bfloat16* Kc,
                          const __nv_bfloat16* Vc, const int64_t* budgets, int Hq, int Hkv,
                          int T, float* out, float* part, size_t part_bytes,
                          cudaStream_t stream) {
  DecodeParams p{};
  p.Hkv = Hkv;
  p.G = Hq / Hkv;
  p.T = T;
  p.nq = p.G * T;
  int64_t total = 0;
  for (int h = 0; h < Hkv; ++h) total += budgets[h];
  p.chunk = decode_chunk_rows(total);
  p.scale2 = 1.4426950408889634f / sqrtf(float(kD));
  p.cu[0] = 0;
  p.wpfx[0] = 0;
  for (int h = 0; h < Hkv; ++h) {
    p.cu[h + 1] = p.cu[h] + int32_t(budgets[h]);
    p.wpfx[h + 1] = p.wpfx[h] + int32_t(ceil_div(budgets[h], p.chunk));
  }
  const int nchunks = p.wpfx[Hkv];
  static_assert(kDMaxChunks >= kDTargetChunks + SGDKV_MAX_KV_HEADS, "chunks per head");
  static_assert(kDWarps * 32 == kD, "one merge thread per column");
  static_assert(kDWarps * 16 * kDPartStride * 4 <= kDWarps * kDWarpBytes, "merge buffer");
  if (size_t(nchunks) * 16 * kDPartStride * sizeof(float) > part_bytes) return cudaErrorInvalidValue;
  const int smem = kDWarps * kDWarpBytes;
  cudaError_t e = cudaFuncSetAttribute(decode_partial_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  if (nchunks > 0) {
    // programmatic dependent launch as well: back-to-back calls (one per layer) overlap,
    // this call's streaming with the previous call's merge
    KernelTimer tk(SGDKV_KERNEL_DECODE, stream);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(nchunks), 1, 1);
    cfg.blockDim = dim3(kDWarps * 32, 1, 1);
    cfg.dynamicSmemBytes = size_t(smem);
    cfg.stream = stream;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_partial_kernel, q, Kc, Vc, p, part);
    if (e != cudaSuccess) return e;
    note_launches(1);
  }
  {
    // programmatic dependent launch: the merge blocks are placed on SMs as soon as there is
    // room (SMs without a partial CTA, then those the partial CTAs leave) and start their
    // work as soon as the partial kernel completes
    KernelTimer tc(SGDKV_KERNEL_DECODE, stream);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(Hkv * p.nq), 1, 1);
    cfg.blockDim = dim3(kDCombThreads, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = nchunks > 0 ? 1 : 0;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_combine_kernel, static_cast<const float*>(part), p, out);
    if (e != cudaSuccess) return e;
    note_launches(1);
  }
  return cudaGetLastError();
}

}  // namespace sgdkv
