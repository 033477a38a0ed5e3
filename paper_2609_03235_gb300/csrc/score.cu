// Window scoring (Section 3.3 / Section 5: cumulative attention of the final observation
// window, SnapKV-style) and max-pool smoothing.
//
// For KV head h the G*W window rows r = g*W + w (query head h*G+g, window position w) are
// contiguous in q_win.  With t_rj = (q_r . k_j) * log2(e)/sqrt(d):
//   pass 1  per row r: m_r = max_j t_rj, Z_r = sum_j 2^(t_rj - m_r) over visible keys,
//           computed per key range and merged into lse_r = m_r + log2 Z_r;
//   pass 2  per key j: raw_j = sum_r 2^(t_rj - lse_r) over rows that see j;
//   pool    scores_j = max raw over [j - pool/2, j + pool/2] clipped to [0, L).
// Row w sees keys j <= L - W + w.
#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float dot_bf16x8(const uint4 a, const uint4 b, float acc) {
  const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
  const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 fa = __bfloat1622float2(pa[i]);
    const float2 fb = __bfloat1622float2(pb[i]);
    acc = fmaf(fa.x, fb.x, acc);
    acc = fmaf(fa.y, fb.y, acc);
  }
  return acc;
}

constexpr int kP1Keys = 32;   // keys staged per step in pass 1

// Pass 1 on CUDA cores: one thread per window row, one CTA per (key range, head).
__global__ void __launch_bounds__(512, 1)
rowstats_simt_kernel(const uint4* __restrict__ q, const uint4* __restrict__ K, int G, int W,
                     int64_t L, int64_t range, float scale2, Ws ws) {
  const int h = blockIdx.y, part = blockIdx.x, r = threadIdx.x, GW = G * W;
  __shared__ uint4 ks[kP1Keys][16];
  uint4 qr[16];
  const bool active = r < GW;
#pragma unroll
  for (int i = 0; i < 16; ++i)
    qr[i] = active ? __ldg(q + (int64_t(h) * GW + r) * 16 + i) : make_uint4(0, 0, 0, 0);
  const int64_t lim = L - W + (active ? r % W : 0);
  const int64_t j0 = int64_t(part) * range;
  const int64_t j1 = j0 + range < L ? j0 + range : L;
  float m = -INFINITY, Z = 0.f;
  for (int64_t jt = j0; jt < j1; jt += kP1Keys) {
    __syncthreads();
    for (int i = threadIdx.x; i < kP1Keys * 16; i += blockDim.x) {
      const int64_t j = jt + i / 16;
      ks[i / 16][i % 16] = j < j1 ? __ldg(K + (int64_t(h) * L + j) * 16 + i % 16)
                                  : make_uint4(0, 0, 0, 0);
    }
    __syncthreads();
    if (!active) continue;
    float t[kP1Keys];
    float tmax = -INFINITY;
#pragma unroll
    for (int kk = 0; kk < kP1Keys; ++kk) {
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) acc = dot_bf16x8(qr[i], ks[kk][i], acc);
      const int64_t j = jt + kk;
      t[kk] = (j < j1 && j <= lim) ? acc * scale2 : -INFINITY;
      tmax = fmaxf(tmax, t[kk]);
    }
    if (tmax == -INFINITY) continue;
    const float mn = fmaxf(m, tmax);
    float z = (m == -INFINITY) ? 0.f : Z * fast_exp2(m - mn);
#pragma unroll
    for (int kk = 0; kk < kP1Keys; ++kk) z += fast_exp2(t[kk] - mn);
    Z = z;
    m = mn;
  }
  if (active)
    ws.partial[(int64_t(h) * kMaxScoreParts + part) * kMaxRows + r] = make_float2(m, Z);
}

// Merges the per-range (m, Z) of every row into lse_r = m_r + log2(Z_r).
__global__ void lse_merge_kernel(int GW, int nparts, Ws ws) {
  const int h = blockIdx.x, r = threadIdx.x;
  if (r >= GW) return;
  const float2* p = ws.partial + int64_t(h) * kMaxScoreParts * kMaxRows + r;
  float M = -INFINITY;
  for (int i = 0; i < nparts; ++i) M = fmaxf(M, p[int64_t(i) * kMaxRows].x);
  float S = 0.f;
  for (int i = 0; i < nparts; ++i) {
    const float2 v = p[int64_t(i) * kMaxRows];
    if (v.x != -INFINITY) S += v.y * fast_exp2(v.x - M);
  }
  ws.lse[h * kMaxRows + r] = M + log2f(S);
}

// Pass 2 on CUDA cores: one thread per key, window rows read from shared memory.
__global__ void __launch_bounds__(128)
accum_simt_kernel(const uint4* __restrict__ q, const uint4* __restrict__ K, int G, int W,
                  int64_t L, float scale2, Ws ws) {
  extern __shared__ uint4 smem[];
  const int h = blockIdx.y, GW = G * W;
  uint4* qs = smem;
  float* lse = reinterpret_cast<float*>(qs + GW * 16);
  for (int i = threadIdx.x; i < GW * 16; i += blockDim.x) qs[i] = __ldg(q + int64_t(h) * GW * 16 + i);
  for (int i = threadIdx.x; i < GW; i += blockDim.x) lse[i] = ws.lse[h * kMaxRows + i];
  __syncthreads();
  const int64_t j = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (j >= L) return;
  uint4 kr[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) kr[i] = __ldg(K + (int64_t(h) * L + j) * 16 + i);
  const int64_t wmin = j - (L - W);   // rows with w >= wmin see key j
  float acc = 0.f;
  for (int r = 0; r < GW; ++r) {
    if (r % W < wmin) continue;
    float d = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) d = dot_bf16x8(qs[r * 16 + i], kr[i], d);
    acc += fast_exp2(fmaf(d, scale2, -lse[r]));
  }
  ws.raw[int64_t(h) * L + j] = acc;
}

__global__ void maxpool_kernel(const float* __restrict__ raw, float* __restrict__ out,
                               int64_t L, int64_t n, int radius) {
  const int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const int64_t j = t % L;
  const float* row = raw + (t - j);
  float m = row[j];
  for (int s = 1; s <= radius; ++s) {
    if (j - s >= 0) m = fmaxf(m, row[j - s]);
    if (j + s < L) m = fmaxf(m, row[j + s]);
  }
  out[t] = m;
}

}  // namespace

cudaError_t launch_score(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                         int64_t L, int W, int pool, float* scores_out, const Ws& ws,
                         cudaStream_t stream) {
  const int G = Hq / Hkv, GW = G * W;
  const float scale2 = kLog2e / sqrtf(float(kD));
  int64_t range = ceil_div(L, kMaxScoreParts);
  range = range < 1024 ? 1024 : ceil_div(range, kP1Keys) * kP1Keys;
  const int nparts = int(ceil_div(L, range));
  const uint4* q4 = reinterpret_cast<const uint4*>(q);
  const uint4* k4 = reinterpret_cast<const uint4*>(K);
  const int p1_threads = int(ceil_div(GW, 32) * 32);
  rowstats_simt_kernel<<<dim3(nparts, Hkv), p1_threads, 0, stream>>>(q4, k4, G, W, L, range,
                                                                     scale2, ws);
  lse_merge_kernel<<<Hkv, p1_threads, 0, stream>>>(GW, nparts, ws);
  const size_t smem = size_t(GW) * 256 + size_t(GW) * 4;
  cudaError_t e = cudaFuncSetAttribute(accum_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  accum_simt_kernel<<<dim3(unsigned(ceil_div(L, 128)), Hkv), 128, smem, stream>>>(q4, k4, G, W,
                                                                                 L, scale2, ws);
  const int64_t n = int64_t(Hkv) * L;
  maxpool_kernel<<<unsigned(ceil_div(n, 256)), 256, 0, stream>>>(ws.raw, scores_out, L, n,
                                                                pool / 2);
  note_launches(4);
  return cudaGetLastError();
}

}  // namespace sgdkv
