// Window scoring on the 5th-generation tensor cores (tcgen05 + TMEM + TMA), sm_103a.
//
// Computes the cumulative window attention of Section 3.3 / Section 5 (SnapKV-style):
//   raw[h][j] = sum_{g<G} sum_{w<W} softmax_j(q[h*G+g][w] . K[h][j] / sqrt(d)),
// window row w seeing keys j <= L - W + w.  With t_rj = (q_r . k_j) * log2(e)/sqrt(d) and
// the G*W window rows r = g*W + w of KV head h (contiguous in q_win):
//
//   pass 1 (score_pass1_tc): D[r][j] = Q_h K_tile^T, window rows on TMEM lanes and keys on
//     columns (MMA N = 128 keys; one 128-column TMEM slot per epilogue warpgroup, each
//     warpgroup owning one row tile).  Every epilogue thread keeps an online (max m_r, sum
//     Z_r = sum 2^(t_rj - m_r)) for its window row over all keys of the key tiles it
//     receives; one partial per row per CTA goes to the workspace.
//   pass 2 (score_pass2_tc): merges the partials into lse_r = m_r + log2 Z_r, then
//     D[j][r] = K_tile Q_h^T (keys on TMEM lanes, rows on columns, Q_h in shared memory);
//     every epilogue thread sums 2^(t_rj - lse_r) for its key over a quarter of the window
//     rows (four warps per key), written to four partial-sum planes of the raw buffer.
//   pool (maxpool_sum_kernel): scores = max-pool of the sum of the four planes.
//
// CTA roles (640 threads): warp 2 lane 0 issues TMA loads (Q_h once, K tiles of 128 keys
// through a ring of shared-memory stages); warp 3 allocates the 512 TMEM columns and its
// elected lane issues the MMAs; warps 4..19 are the epilogue (four per TMEM lane quarter);
// warps 0 and 1 idle, so that the control warps share sub-partitions with the lane
// quarters that carry less epilogue work.  An epilogue warp loads its TMEM columns of a
// slot block by block, summing one block while the next is in flight, and releases the
// slot once its last block has landed, so the MMAs of the next slot use overlap the rest of
// the arithmetic.  Pass 1 has four slots of 128 columns (one per epilogue warpgroup), pass 2
// two of 256 shared by all sixteen epilogue warps.  Each CTA owns one KV head and claims its key tiles from a counter shared by the
// head's CTAs.  Every wait on an mbarrier is bounded in time:
// on expiry the kernel records SGDKV_ERR_TIMEOUT, all roles leave their loops, in-flight
// copies and MMAs are drained (again bounded) and TMEM is freed.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "sgdkv_internal.cuh"

namespace sgdkv {
namespace {

// Warp roles.  Warp w runs on SM sub-partition w % 4 and reaches TMEM lanes 32 * (w % 4)..
// The producer and the MMA warp sit on sub-partitions 2 and 3: with G*W rows padded to
// 128-row tiles, the extra (partial) row tile of pass 1 lands on lane quarters 0 and 1, so
// the four sub-partitions carry about the same load.  Warps 0 and 1 have no role.
constexpr int kProducerWarp = 2;
constexpr int kMmaWarp = 3;
constexpr int kFirstEpiWarp = 4;                  // warps 4..19: epilogue, four per quarter
constexpr int kThreads = 640;                     // 20 warps
constexpr int kEpiWarps = 16;
constexpr int kMaxRegs = 96;   // 5 warps x 96 x 32 fit one 16K-register SM sub-partition
constexpr int kTileKeys = 128;
constexpr uint32_t kTmemCols = 512;
constexpr int kStageBytes = kTileKeys * 256;      // 32 KB: two 128-byte column halves
constexpr int kHalfBytes = kTileKeys * 128;       // 16 KB
constexpr int kMaxStages = 8;
constexpr int kTmemSlots = 4;                     // TMEM slots (pass 1: 4 x 128 columns, pass 2: 2 x 256)
constexpr int kNumBars = 2 * kMaxStages + 2 * kTmemSlots + 3;   // kfull kempty tfull tempty qfull drain never
constexpr int kCtlBytes = 512;                    // barriers, TMEM address, abort flag, tile ids
static_assert(kNumBars * 8 + 8 + (kMaxStages + kTmemSlots + 1) * 4 <= kCtlBytes, "control block");
constexpr int kSmemLimit = 232448;                // opt-in dynamic shared memory per CTA
constexpr int kQBoxRows = 32;                     // TMA box height for Q rows (pass 2)
constexpr uint32_t kFlagStallMma = 1u;            // test hook: MMA thread waits on `never`
constexpr float kLog2e = 1.4426950408889634f;
constexpr uint64_t kDrainNs = 1000000000ull;      // bound on cleanup waits after an abort

struct TcParams {
  int Hkv, G, W, GW;
  int64_t L;
  int T;          // key tiles (of 128) per head
  int cph;        // CTAs per head (each claims key tiles of its head until none are left)
  int nrt;        // window-row tiles of 128 = ceil(GW / 128)
  int nstages;    // K ring depth
  int nparts;     // pass 2: partial slots per head written by pass 1
  float scale2;   // log2(e) / sqrt(d)
  int causal;     // 1: window row w sees keys <= L - W + w; 0: every row sees all L keys
  int agg;        // SGDKV_SCORE_AGG_* >> 1: 0 sum over the group, 1 IPT max, 2 IPT mean, 3 IPT only
  const float* head_w;   // IPT modes: summarization score per query head [Hq]
  int det;        // SGDKV_SCORE_DETERMINISTIC: pass 1 takes fixed key tiles per CTA
  uint64_t wait_ns;
  uint32_t flags;
};

// ---------------------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]),
                 "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
                 "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]),
                 "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive2(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], 2;" ::"r"(bar) : "memory");
}
// The waiting thread is suspended until the phase completes or kSuspendNs elapse, so a
// waiting warp does not take issue slots from the working warps of its sub-partition.
constexpr uint32_t kSuspendNs = 20000;
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "n"(kSuspendNs)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits for the phase of `bar` with the given parity; false if the CTA aborted or the wait
// ran past limit_ns (then the timeout is recorded and the CTA-wide abort flag raised).
__device__ __noinline__ bool bwait_slow(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                        uint64_t limit_ns, uint32_t* status) {
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try(bar, parity)) return true;
    if ((it & 3u) == 0) {
      if (*abort_flag) return false;
      if (global_ns() - t0 > limit_ns) {
        record_error(status, SGDKV_ERR_TIMEOUT);
        *abort_flag = 1;
        return false;
      }
    }
  }
}
// Completed phases (the common case on the critical path) return after one test, inline.
__device__ __forceinline__ bool bwait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                      uint64_t limit_ns, uint32_t* status) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok ? true : bwait_slow(bar, parity, abort_flag, limit_ns, status);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// The same with an L2 cache policy (createpolicy) for the copied lines.
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap* map, int x,
                                                 int y, uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
// L2 policy of lines read for the last time: first to be evicted.
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// Shared-memory matrix descriptor (K-major operand, 128-byte swizzle, rows of 128 bytes in
// 8-row atoms of 1024 bytes: the layout a TMA box {64 bf16, rows} with SWIZZLE_128B writes),
// kept as two 32-bit words.  High word: stride between 8-row groups 1024 B, descriptor
// version 1, SWIZZLE_128B.  Low word: start address / 16 (< 2^14 for shared memory) and the
// leading-dimension field set to 1 (unused by this layout); an operand advanced by `bytes`
// has low word + bytes / 16.
constexpr uint32_t kDescHi = (1024u >> 4) | (1u << 14) | (2u << 29);
__device__ __forceinline__ uint32_t desc_lo(uint32_t saddr) { return (saddr >> 4) | (1u << 16); }
// Instruction descriptor, kind::f16: bf16 A and B (K-major), fp32 accumulator, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(N >> 3) << 17) | (uint32_t(M >> 4) << 24);
}
// One lane of the converged warp (the MMA warp runs its loop with all 32 lanes, so the
// operands stay warp-uniform; the elected lane alone issues MMAs, commits and arrivals).
__device__ __forceinline__ uint32_t elect_one() {
  uint32_t e;
  asm volatile(
      "{\n\t.reg .pred P;\n\telect.sync _|P, 0xffffffff;\n\tselp.u32 %0, 1, 0, P;\n\t}"
      : "=r"(e));
  return e;
}
// tcgen05.mma kind::f16 from low descriptor words, issued by the lane with leader != 0; ACC
// is a compile-time accumulate flag.
template <int ACC>
__device__ __forceinline__ void umma_lo(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo,
                                        uint32_t idesc, uint32_t leader) {
  asm volatile(
      "{\n\t.reg .b64 ad, bd;\n\t.reg .pred p, l;\n\t"
      "mov.b64 ad, {%1, %4};\n\tmov.b64 bd, {%2, %4};\n\t"
      "setp.ne.b32 p, %5, 0;\n\tsetp.ne.b32 l, %6, 0;\n\t"
      "@l tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_lo), "r"(b_lo), "r"(idesc), "r"(kDescHi), "n"(ACC), "r"(leader)
      : "memory");
}
// The 8 k steps (16 columns each of the two 64-column halves) of one 128 x N x 128 MMA:
// A and B advance 32 B per step within a half and jump by their half strides.
__device__ __forceinline__ void umma_k128(uint32_t d_tmem, uint32_t a_lo, uint32_t a_half,
                                          uint32_t b_lo, uint32_t b_half, uint32_t idesc,
                                          uint32_t leader) {
  umma_lo<0>(d_tmem, a_lo, b_lo, idesc, leader);
#pragma unroll
  for (int k = 1; k < 8; ++k) {
    const uint32_t ka = (k >> 2) * a_half + (k & 3) * 2, kb = (k >> 2) * b_half + (k & 3) * 2;
    umma_lo<1>(d_tmem, a_lo + ka, b_lo + kb, idesc, leader);
  }
}
__device__ __forceinline__ void umma_commit(uint32_t bar, uint32_t leader) {
  asm volatile(
      "{\n\t.reg .pred l;\n\tsetp.ne.b32 l, %1, 0;\n\t"
      "@l tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(bar),
      "r"(leader)
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

#define SGDKV_LD_REGS32(r)                                                                   \
  "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),       \
      "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), \
      "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),          \
      "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),          \
      "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])

// 32 consecutive fp32 TMEM columns of this thread's lane (32x32b shape, x32).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : SGDKV_LD_REGS32(r)
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
// Waits for this thread's TMEM loads, with the registers of the load it completes passed
// through it: code that reads them cannot be scheduled above the wait while a later load is
// still in flight.
__device__ __forceinline__ void tmem_wait_ld(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                 "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                 "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// Packed fp32 pairs (sm_100 family f32x2 arithmetic: one instruction for two lanes).
__device__ __forceinline__ uint64_t pk(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ uint64_t pku(uint32_t lo, uint32_t hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ void upk(uint64_t r, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(r));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// 2^(v*s - n) for two lanes, accumulated into the packed pair acc.
__device__ __forceinline__ uint64_t acc_exp2(uint64_t acc, uint32_t v0, uint32_t v1, uint64_t s2,
                                             uint64_t neg) {
  float x0, x1;
  upk(fma2(pku(v0, v1), s2, neg), x0, x1);
  return add2(acc, pk(ex2(x0), ex2(x1)));
}
__device__ __forceinline__ float hsum(uint64_t a, uint64_t b) {
  float a0, a1, b0, b1;
  upk(a, a0, a1);
  upk(b, b0, b1);
  return (a0 + a1) + (b0 + b1);
}

// Tile ids handed between roles through shared memory: explicit shared-space accesses (a
// volatile access through a generic pointer compiles to a system-scope load), ordered by
// the mbarrier arrive (release) and wait (acquire) around them.
__device__ __forceinline__ int ld_tile(const volatile int* p) {
  int v;
  asm volatile("ld.volatile.shared.s32 %0, [%1];" : "=r"(v) : "r"(smem_u32((const void*)p)) : "memory");
  return v;
}
__device__ __forceinline__ void st_tile(volatile int* p, int v) {
  asm volatile("st.volatile.shared.s32 [%0], %1;" ::"r"(smem_u32((const void*)p)), "r"(v) : "memory");
}

// ---------------------------------------------------------------------------------------
// ---------------------------------------------------------------------------------------
// Shared pieces of both passes
// ---------------------------------------------------------------------------------------
struct Smem {
  uint8_t* q;          // 2 column halves x qrows x 128 B (pass 1: padded to row tiles)
  uint8_t* k;          // nstages x 32 KB
  uint64_t* bars;      // kNumBars
  uint32_t* tmem_slot;
  int* abort_flag;
  volatile int* stile; // [kMaxStages] key tile held by each K stage (-1: no more tiles)
  volatile int* utile; // [kTmemSlots] key tile whose products fill each TMEM slot (-1: done)
  volatile uint32_t* claims;   // the producer's last claim (see produce)
  float* tail;         // pass 2: -lse2[kMaxRows] (16-byte aligned)
  int qrows;
};

__device__ __forceinline__ Smem carve(uint8_t* base, int qrows, int nstages) {
  Smem s;
  s.qrows = qrows;
  s.q = base;
  s.k = base + 2 * qrows * 128;
  uint8_t* ctl = s.k + nstages * kStageBytes;
  s.bars = reinterpret_cast<uint64_t*>(ctl);
  s.tmem_slot = reinterpret_cast<uint32_t*>(ctl + kNumBars * 8);
  s.abort_flag = reinterpret_cast<int*>(ctl + kNumBars * 8 + 4);
  s.stile = reinterpret_cast<int*>(ctl + kNumBars * 8 + 8);
  s.utile = s.stile + kMaxStages;
  s.claims = reinterpret_cast<volatile uint32_t*>(s.utile + kTmemSlots);
  s.tail = reinterpret_cast<float*>(ctl + kCtlBytes);
  return s;
}
__device__ __forceinline__ uint32_t bar_kfull(const Smem& s, int i) { return smem_u32(s.bars + i); }
__device__ __forceinline__ uint32_t bar_kempty(const Smem& s, int i) { return smem_u32(s.bars + kMaxStages + i); }
__device__ __forceinline__ uint32_t bar_tfull(const Smem& s, int i) { return smem_u32(s.bars + 2 * kMaxStages + i); }
__device__ __forceinline__ uint32_t bar_tempty(const Smem& s, int i) { return smem_u32(s.bars + 2 * kMaxStages + kTmemSlots + i); }
__device__ __forceinline__ uint32_t bar_qfull(const Smem& s) { return smem_u32(s.bars + 2 * kMaxStages + 2 * kTmemSlots); }
__device__ __forceinline__ uint32_t bar_drain(const Smem& s) { return smem_u32(s.bars + 2 * kMaxStages + 2 * kTmemSlots + 1); }
__device__ __forceinline__ uint32_t bar_never(const Smem& s) { return smem_u32(s.bars + 2 * kMaxStages + 2 * kTmemSlots + 2); }

// Barrier init, TMEM allocation; returns the TMEM base address (all threads).
// nslots TMEM slots whose tempty barriers expect `consumers` warp arrivals each.
__device__ __forceinline__ uint32_t setup(const Smem& s, int nstages, uint32_t qfull_count,
                                          int nslots, uint32_t consumers) {
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < nstages; ++i) {
      mbar_init(bar_kfull(s, i), 1);
      mbar_init(bar_kempty(s, i), 1);
    }
    // tfull: one plain arrive of the MMA thread (publishing utile) + its MMA commit
    for (int i = 0; i < nslots; ++i) {
      mbar_init(bar_tfull(s, i), 2);
      mbar_init(bar_tempty(s, i), consumers);
    }
    mbar_init(bar_qfull(s), qfull_count);
    mbar_init(bar_drain(s), 1);
    mbar_init(bar_never(s), 1);
    *s.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(s.tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  return *s.tmem_slot;
}

__device__ __forceinline__ void teardown(uint32_t tmem) {
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if ((threadIdx.x >> 5) == kMmaWarp) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

// Producer thread, once its last claim has returned: the head's last CTA to get here resets
// the head's tile counter (and the finish count) for the next launch.
__device__ __forceinline__ void finish_claims(uint32_t* counter, uint32_t* finished, int cph) {
  __threadfence();
  if (atomicAdd(finished, 1u) == uint32_t(cph - 1)) {
    atomicExch(counter, 0u);
    atomicExch(finished, 0u);
  }
}

// TMA producer (one thread): key tiles of head h claimed one at a time from the head's
// counter (shared by the head's CTAs; `first` is the claim made at kernel entry, the next
// claim is made while the current tile's stage is awaited) until none are left -- or, with
// stride > 0, the fixed tiles first, first + stride, ... (no counter) -- and the Q
// rows of head h once, right after the first key tile (which comes from HBM, the Q rows from
// L2); the stage after the last tile carries tile id -1 and no data.  Once its last claim
// has returned the thread counts the CTA's claims finished (finish_claims), while the CTA's
// last tiles are still being consumed.  second (pass 2): pass 2 reads the keys pass 1 has just
// read, so it takes a head's tiles from the last one down, starting on the tiles pass 1
// loaded last, which are still in L2, and loads them evict-first (nothing reads them after
// pass 2), so that its misses do not push out the tiles it has yet to reach.
__device__ void produce(const Smem& s, const CUtensorMap* tm_q, const CUtensorMap* tm_k,
                        const TcParams& p, int h, uint32_t* counter, uint32_t* finished,
                        uint32_t first, uint32_t stride, bool second, uint32_t* status) {
  volatile int* ab = s.abort_flag;
  bool q_issued = false;
  auto load_q = [&] {
    mbar_expect_tx(bar_qfull(s), uint32_t(2 * s.qrows * 128));
    for (int c = 0; c < 2; ++c)
      for (int b = 0; b < s.qrows / kQBoxRows; ++b)
        tma_load_2d(smem_u32(s.q + (c * s.qrows + b * kQBoxRows) * 128), tm_q, 64 * c,
                    h * p.GW + kQBoxRows * b, bar_qfull(s));
    q_issued = true;
  };
  int issued[kMaxStages];
  for (int i = 0; i < kMaxStages; ++i) issued[i] = 0;
  const uint64_t k_policy = second ? l2_evict_first() : 0;
  uint32_t next = first;                        // the next claim overlaps the stage wait
  for (int n = 0;; ++n) {
    const int st = n % p.nstages;
    const int use = n / p.nstages;
    const uint32_t claim = next;
    const uint32_t tile =
        second && claim < uint32_t(p.T) ? uint32_t(p.T) - 1u - claim : claim;
    if (claim < uint32_t(p.T)) next = stride ? claim + stride : atomicAdd(counter, 1u);
    if (!bwait(bar_kempty(s, st), (use & 1) ^ 1, ab, p.wait_ns, status)) break;
    if (tile >= uint32_t(p.T)) {
      st_tile(s.stile + st, -1);
      mbar_arrive(bar_kfull(s, st));            // releases the id; no copy in flight
      if (!q_issued) load_q();
      break;
    }
    st_tile(s.stile + st, int(tile));
    mbar_expect_tx(bar_kfull(s, st), kStageBytes);
    const int row = int(int64_t(h) * p.L + int64_t(tile) * kTileKeys);
    for (int c = 0; c < 2; ++c) {
      const uint32_t dst = smem_u32(s.k + st * kStageBytes + c * kHalfBytes);
      if (second)
        tma_load_2d_hint(dst, tm_k, 64 * c, row, bar_kfull(s, st), k_policy);
      else
        tma_load_2d(dst, tm_k, 64 * c, row, bar_kfull(s, st));
    }
    issued[st] = use + 1;
    if (!q_issued) load_q();
  }
  // The claim still in flight after an abort is waited for by this store; then every claim
  // of the CTA has reached the counter.
  *s.claims = next;
  finish_claims(counter, finished, p.cph);
  if (*ab) {
    // Drain: every copy this thread started must have landed before the CTA exits.
    volatile int no_abort = 0;
    if (q_issued) bwait(bar_qfull(s), 0, &no_abort, kDrainNs, status);
    for (int st = 0; st < p.nstages; ++st)
      if (issued[st] > 0)
        bwait(bar_kfull(s, st), (issued[st] - 1) & 1, &no_abort, kDrainNs, status);
  }
}

// MMA warp (all lanes): bwait with one outcome for the whole warp.
__device__ __forceinline__ bool wwait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                      uint64_t limit_ns, uint32_t* status) {
  return __all_sync(0xffffffffu, bwait(bar, parity, abort_flag, limit_ns, status));
}

// MMA warp, start of its work: the optional stall hook (a wait on a barrier nothing
// arrives on, to exercise the timeout path), then the wait for the Q rows.
__device__ bool mma_start(const Smem& s, const TcParams& p, uint32_t* status) {
  volatile int* ab = s.abort_flag;
  if ((p.flags & kFlagStallMma) && !wwait(bar_never(s), 0, ab, p.wait_ns, status)) return false;
  return wwait(bar_qfull(s), 0, ab, p.wait_ns, status);
}

// Publishes the key tile of a TMEM slot use to the epilogue (the plain arrive on tfull
// releases the store; the MMA commit is the barrier's second arrival).  Tile -1 ends the
// epilogue's loop: both arrivals are made here.
__device__ __forceinline__ void publish_slot(const Smem& s, int slot, int tile, uint32_t leader) {
  if (!leader) return;
  st_tile(s.utile + slot, tile);
  if (tile < 0) mbar_arrive2(bar_tfull(s, slot));
  else mbar_arrive(bar_tfull(s, slot));
}


// MMA warp, after an abort: a commit arrives on `drain` once every MMA the warp issued has
// completed, so TMEM is not released under a running MMA.
__device__ void mma_drain(const Smem& s, uint32_t leader, uint32_t* status) {
  umma_commit(bar_drain(s), leader);
  volatile int no_abort = 0;
  bwait(bar_drain(s), 0, &no_abort, kDrainNs, status);
  __syncwarp();
}

// ---------------------------------------------------------------------------------------
// Pass 1: per window row, online (max, sum of 2^(t - max)) over the CTA's key range
// ---------------------------------------------------------------------------------------
template <int N>
__device__ __forceinline__ float chunk_sum(const uint32_t (&v)[N], float s2, float m) {
  const uint64_t s22 = pk(s2, s2), nm2 = pk(-m, -m);
  uint64_t a0 = 0, a1 = 0;
#pragma unroll
  for (int e = 0; e < N; e += 4) {
    a0 = acc_exp2(a0, v[e], v[e + 1], s22, nm2);
    a1 = acc_exp2(a1, v[e + 2], v[e + 3], s22, nm2);
  }
  return hsum(a0, a1);
}

// Folds N logits of one row (raw dot products in v, keys kb .. kb+N-1) into (m, Z), both in
// log2 units.  Common case: the running max already bounds the chunk to within 2^32, so
// the chunk is summed against it directly; otherwise (first chunk, a much larger logit,
// masked lanes) the chunk max is taken first and Z is rescaled.
template <int N>
__device__ __forceinline__ void online_fold(uint32_t (&v)[N], int kb, bool edge, int lim,
                                            float s2, float& m, float& Z) {
  if (edge) {
#pragma unroll
    for (int e = 0; e < N; ++e)
      if (kb + e > lim) v[e] = 0xff800000u;             // -inf: key not visible to this row
  }
  float zc = chunk_sum<N>(v, s2, m);
  if (!(zc < 4294967296.f)) {
    float mx = -INFINITY;
#pragma unroll
    for (int e = 0; e < N; ++e) mx = fmaxf(mx, __uint_as_float(v[e]));
    if (mx == -INFINITY) return;
    const float mn = fmaxf(m, mx * s2);
    Z = (m == -INFINITY) ? 0.f : Z * ex2(m - mn);
    m = mn;
    zc = chunk_sum<N>(v, s2, m);
  }
  Z += zc;
}

// NRT: row tiles of 128 window rows (1..4).  Q_h (padded to NRT x 128 rows) sits in shared
// memory as the MMA's A operand, K tiles are B.  TMEM holds four slots of 128 columns, one per
// epilogue warpgroup (the four warps wi of the lane quarters): warpgroup w takes row tile
// w % NRT of the key tiles n with n % NB == w / NRT (NB = 4 / NRT warpgroups share a row
// tile, taking alternate key tiles; for NRT = 3 warpgroup 3 has no work).  Per key tile the
// MMA fills the slots of that tile's warpgroups (M = 128 rows, N = 128 keys), and each warp
// folds all 128 keys into the (max, sum) of its 32 rows: one slot wait and one release per
// key tile, one running (m, Z) per thread.
template <int NRT>
__global__ void __maxnreg__(kMaxRegs)
score_pass1_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               TcParams p, Ws ws) {
  constexpr int NB = 4 / NRT;                  // key-tile phases (warpgroups per row tile)
  constexpr int NWG = NRT * NB;                // warpgroups with work
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {
    if (threadIdx.x == 0) record_error(ws.status, SGDKV_ERR_INTERNAL);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // heads interleaved over the block indices: CTAs that wait for an SM held by another
  // kernel are spread across the heads instead of delaying one head's whole share
  const int h = blockIdx.x % p.Hkv, ci = blockIdx.x / p.Hkv;
  uint32_t* counter = ws.sched + h;
  // the first claim's round trip overlaps the barrier and TMEM setup; with fixed tiles
  // (p.det) CTA ci takes tiles ci, ci + cph, ... and the counter is not used
  const uint32_t first = p.det ? uint32_t(ci)
                               : (warp == kProducerWarp && lane == 0 ? atomicAdd(counter, 1u) : 0u);
  const Smem s = carve(smem_raw, NRT * 128, p.nstages);
  const uint32_t tmem = setup(s, p.nstages, 1, kTmemSlots, 4);
  volatile int* ab = s.abort_flag;

  if (warp == kProducerWarp) {
    if (lane == 0)
      produce(s, &tm_q, &tm_k, p, h, counter, ws.sched + SGDKV_MAX_KV_HEADS + h, first,
              p.det ? uint32_t(p.cph) : 0u, false, ws.status);
  } else if (warp == kMmaWarp) {
    const uint32_t leader = elect_one();
    const uint32_t idesc = idesc_bf16(128, kTileKeys);
    bool ok = mma_start(s, p, ws.status);
    const uint32_t q_lo = desc_lo(smem_u32(s.q)), qhalf = uint32_t(s.qrows * 128);
    int fills[kTmemSlots] = {0, 0, 0, 0};        // uses of each slot so far
    for (int n = 0; ok; ++n) {
      const int st = n % p.nstages;
      if (!(ok = wwait(bar_kfull(s, st), (n / p.nstages) & 1, ab, p.wait_ns, ws.status))) break;
      tc_fence_after();
      const int tile = ld_tile(s.stile + st);
      const uint32_t k_lo = desc_lo(smem_u32(s.k + st * kStageBytes));
      const int ph = n % NB;
#pragma unroll
      for (int w = 0; w < NWG; ++w) {
        if (tile >= 0 && w / NRT != ph) continue;   // the end (tile -1) goes to every slot
        if (!(ok = wwait(bar_tempty(s, w), (fills[w] & 1) ^ 1, ab, p.wait_ns, ws.status))) break;
        tc_fence_after();
        publish_slot(s, w, tile, leader);
        ++fills[w];
        if (tile < 0) continue;
        umma_k128(tmem + uint32_t(w * kTileKeys), q_lo + uint32_t(w % NRT) * (kHalfBytes >> 4),
                  qhalf >> 4, k_lo, kHalfBytes >> 4, idesc, leader);
        umma_commit(bar_tfull(s, w), leader);
      }
      if (tile < 0 || !ok) break;
      umma_commit(bar_kempty(s, st), leader);
    }
    if (!ok) mma_drain(s, leader, ws.status);
  } else if (warp >= kFirstEpiWarp) {
    const int q = warp & 3, wi = (warp - kFirstEpiWarp) >> 2;
    const int rt = wi % NRT, ph = wi / NRT;
    const int r = rt * 128 + 32 * q + lane;              // this thread's window row
    const bool valid = wi < NWG && rt * 128 + 32 * q < p.GW;   // warp-uniform
    // keys above a row's limit are masked; lim_base: the lowest limit of any row
    const int lim_base = p.causal ? int(p.L - p.W) : int(p.L - 1);   // Hkv * L < 2^31
    const int lim = p.causal ? lim_base + r % p.W : lim_base;
    float m = -INFINITY, Z = 0.f;
    if (wi < NWG) {
      const uint32_t tf = bar_tfull(s, wi), te = bar_tempty(s, wi);
      const uint32_t tb = tmem + (uint32_t(32 * q) << 16) + uint32_t(wi * kTileKeys);
      for (int c = 0;; ++c) {
        if (!bwait(tf, c & 1, ab, p.wait_ns, ws.status)) break;
        tc_fence_after();
        const int tile = ld_tile(s.utile + wi);
        if (tile < 0) break;                             // no more tiles
        auto release = [&] {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(te);
        };
        if (!valid) {
          release();
          continue;
        }
        // 4 blocks of 32 keys: block b + 1 in flight while block b is folded; the slot is
        // released once the last block has landed.
        const int kb = tile * kTileKeys;
        uint32_t v[2][32];
        tmem_ld32(tb, v[0]);
        tmem_wait_ld(v[0]);
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          if (b < 3) tmem_ld32(tb + uint32_t(32 * (b + 1)), v[(b + 1) & 1]);
          else release();
          online_fold<32>(v[b & 1], kb + 32 * b, kb + 32 * b + 31 > lim_base, lim, p.scale2, m,
                          Z);
          if (b < 3) tmem_wait_ld(v[(b + 1) & 1]);
        }
      }
    }
    // The NB warpgroups of a row tile merge their (m, Z) in shared memory, in the K ring:
    // once every epilogue warp has seen the end of its slot, the last MMA of every slot has
    // completed and the ring is idle.  One partial per row per CTA.
    float2* red = reinterpret_cast<float2*>(s.k);           // [NB][kMaxRows]
    if (NB > 1) {
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
      if (valid && !*ab) red[ph * kMaxRows + r] = make_float2(m, Z);
      asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
    }
    if (valid && ph == 0 && !*ab) {
      float M = m, S = Z;
      if (NB > 1) {
        M = -INFINITY;
#pragma unroll
        for (int i = 0; i < NB; ++i) M = fmaxf(M, red[i * kMaxRows + r].x);
        S = 0.f;
#pragma unroll
        for (int i = 0; i < NB; ++i) {
          const float2 e = red[i * kMaxRows + r];
          if (e.x != -INFINITY) S += e.y * ex2(e.x - M);
        }
      }
      ws.partial[(int64_t(h) * kMaxScoreParts + ci) * kMaxRows + r] = make_float2(M, S);
    }
  }
  teardown(tmem);
}

// ---------------------------------------------------------------------------------------
// Pass 2: per key, sum over window rows of 2^(t - lse)
// ---------------------------------------------------------------------------------------
// One pass-2 slot use in the usual case: no key of the tile is masked and the warp's NB
// blocks of 16 columns sit at li0, li0 + 4, ... (all offsets but li0 fixed at compile time,
// so the loop has no branches).  Block k + 1 is loaded while block k is summed; the slot is
// released once the last block has landed.
template <int NB>
__device__ __forceinline__ void p2_use(uint32_t tb, int li0, const float* lse_c, uint64_t s22,
                                       uint32_t tempty, int lane, uint64_t& a0, uint64_t& a1) {
  uint32_t v[2][16];
  tmem_ld16(tb + uint32_t(li0 * 16), v[0]);
  tmem_wait_ld(v[0]);
#pragma unroll
  for (int k = 0; k < NB; ++k) {
    if (k + 1 < NB) {
      tmem_ld16(tb + uint32_t((li0 + 4 * (k + 1)) * 16), v[(k + 1) & 1]);
    } else {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty);
    }
    const float4* nl = reinterpret_cast<const float4*>(lse_c + (li0 + 4 * k) * 16);
#pragma unroll
    for (int e = 0; e < 16; e += 4) {
      const float4 b = nl[e >> 2];
      a0 = acc_exp2(a0, v[k & 1][e], v[k & 1][e + 1], s22, pk(b.x, b.y));
      a1 = acc_exp2(a1, v[k & 1][e + 2], v[k & 1][e + 3], s22, pk(b.z, b.w));
    }
    if (k + 1 < NB) tmem_wait_ld(v[(k + 1) & 1]);
  }
}

// PERG (IPT max aggregation): each epilogue warp takes the 16-column blocks of whole query
// heads (head g goes to the warps with wi = g % 4, W % 16 == 0, G <= 8), keeps a sum per
// head and writes the larger of its (at most two) weighted head sums; the four planes are
// then combined by max instead of sum.
template <bool PERG>
__global__ void __maxnreg__(kMaxRegs)
score_pass2_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               TcParams p, Ws ws) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {
    if (threadIdx.x == 0) record_error(ws.status, SGDKV_ERR_INTERNAL);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.x % p.Hkv;             // heads interleaved, as in pass 1
  uint32_t* counter = ws.sched + 2 * SGDKV_MAX_KV_HEADS + h;
  const uint32_t first = warp == kProducerWarp && lane == 0 ? atomicAdd(counter, 1u) : 0u;
  const Smem s = carve(smem_raw, p.GW, p.nstages);
  float* lse2 = s.tail;                          // [kMaxRows], negated
  const uint32_t tmem = setup(s, p.nstages, 1, 2, kEpiWarps);
  volatile int* ab = s.abort_flag;
  const int nch = p.GW > 256 ? 2 : 1;            // N chunks of the window rows per tile
  const int nn = p.GW / nch;                     // MMA N

  if (warp == kProducerWarp) {
    if (lane == 0)
      produce(s, &tm_q, &tm_k, p, h, counter, ws.sched + 3 * SGDKV_MAX_KV_HEADS + h, first, 0u,
              true, ws.status);
  } else if (warp == kMmaWarp) {
    const uint32_t leader = elect_one();
    const uint32_t idesc = idesc_bf16(128, nn);
    bool ok = mma_start(s, p, ws.status);
    const uint32_t q_lo = desc_lo(smem_u32(s.q)), qhalf = uint32_t(s.qrows * 128);
    for (int n = 0; ok; ++n) {
      const int st = n % p.nstages;
      if (!(ok = wwait(bar_kfull(s, st), (n / p.nstages) & 1, ab, p.wait_ns, ws.status))) break;
      tc_fence_after();
      const int tile = ld_tile(s.stile + st);
      const uint32_t k_lo = desc_lo(smem_u32(s.k + st * kStageBytes));
      for (int c = 0; c < nch; ++c) {
        const int u = n * nch + c, slot = u & 1;
        if (!(ok = wwait(bar_tempty(s, slot), ((u >> 1) & 1) ^ 1, ab, p.wait_ns, ws.status)))
          break;
        tc_fence_after();
        publish_slot(s, slot, tile, leader);
        if (tile < 0) break;
        umma_k128(tmem + uint32_t(slot * 256), k_lo, kHalfBytes >> 4,
                  q_lo + uint32_t(c * nn) * (128 >> 4), qhalf >> 4, idesc, leader);
        umma_commit(bar_tfull(s, slot), leader);
      }
      if (tile < 0) break;
      if (ok) umma_commit(bar_kempty(s, st), leader);
    }
    if (!ok) mma_drain(s, leader, ws.status);
  } else if (warp >= kFirstEpiWarp) {
    const int ew = warp - kFirstEpiWarp, q = warp & 3, wi = ew >> 2;
    // Merge pass-1 partials of every window row into lse2 (log2 units): one online pass,
    // twenty independent loads in flight per step.
    for (int r = ew * 32 + lane; r < p.GW; r += kEpiWarps * 32) {
      const float2* pp = ws.partial + int64_t(h) * kMaxScoreParts * kMaxRows + r;
      float M = -INFINITY, S = 0.f;
      constexpr int kB = 20;
      for (int i0 = 0; i0 < p.nparts; i0 += kB) {
        float2 v[kB];
#pragma unroll
        for (int i = 0; i < kB; ++i)
          v[i] = i0 + i < p.nparts ? __ldcg(pp + int64_t(i0 + i) * kMaxRows)
                                   : make_float2(-INFINITY, 0.f);
#pragma unroll
        for (int i = 0; i < kB; ++i) {
          if (v[i].x == -INFINITY) continue;
          const float mn = fmaxf(M, v[i].x);
          S = (M == -INFINITY ? 0.f : S * ex2(M - mn)) + v[i].y * ex2(v[i].x - mn);
          M = mn;
        }
      }
      float bias = 0.f;                           // log2 of the row's weight in the sum
      if (p.agg != 0) {
        const int G = p.GW / p.W, g = r / p.W;
        const float* wq = p.head_w + h * G;       // the group's summarization scores
        auto ok_w = [&](float x) { return x >= 0.f && x < INFINITY; };
        const float w = wq[g];
        if (!ok_w(w)) record_error(ws.status, SGDKV_ERR_INVALID_ARG);
        if (p.agg == 3) {                         // only the group's top head (lower g on ties)
          int best = 0;
          float bw = ok_w(wq[0]) ? wq[0] : -1.f;
          for (int i = 1; i < G; ++i) {
            const float x = ok_w(wq[i]) ? wq[i] : -1.f;
            if (x > bw) {
              bw = x;
              best = i;
            }
          }
          bias = g == best ? 0.f : -INFINITY;
        } else {
          const float x = ok_w(w) ? (p.agg == 2 ? w / float(G) : w) : 0.f;
          bias = x > 0.f ? log2f(x) : -INFINITY;
        }
      }
      lse2[r] = bias - (M + log2f(S));            // stored negated: the bias of the FMA
    }
    asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
    const uint64_t s22 = pk(p.scale2, p.scale2);
    // The 4 warps of lane quarter q share its 32 keys; the window rows of every N chunk
    // are dealt to them in blocks of 16 columns, round robin over the whole tile (PERG: by
    // query head).
    const int gpc = nn / 16;                     // 16-column blocks per chunk (<= 16)
    float* raw_out = ws.raw + int64_t(wi) * p.Hkv * p.L + int64_t(h) * p.L;
    const int lim_base = p.causal ? int(p.L - p.W) : int(p.L - 1);   // lowest row limit
    // this warp's first block and block count in chunks 0 and 1 (loop invariants)
    const int li0_0 = wi, li0_1 = (((wi - gpc) % 4) + 4) % 4;
    const int ng_0 = li0_0 < gpc ? (gpc - li0_0 + 3) / 4 : 0;
    const int ng_1 = li0_1 < gpc ? (gpc - li0_1 + 3) / 4 : 0;
    bool ok = true;
    for (int n = 0; ok; ++n) {
      int j = 0;
      uint64_t acc0 = 0, acc1 = 0, acc2 = 0, acc3 = 0;   // PERG: acc0/1 head slot 0, acc2/3 slot 1
      for (int c = 0; c < nch; ++c) {
        const int u = n * nch + c, slot = u & 1;
        if (!(ok = bwait(bar_tfull(s, slot), (u >> 1) & 1, ab, p.wait_ns, ws.status))) break;
        tc_fence_after();
        const int tile = ld_tile(s.utile + slot);
        if (tile < 0) {
          ok = false;                              // no more tiles
          break;
        }
        const int key0 = tile * kTileKeys;
        j = key0 + 32 * q + lane;
        const bool masked = key0 + kTileKeys - 1 > lim_base;
        // this warp's blocks of chunk c (at most 4): block k is li0 + 4k (PERG: blk[k])
        int blk[4], ng = 0, li0 = 0;
        if (PERG) {
          for (int b = 0; b < gpc && ng < 4; ++b)
            if (((c * nn + 16 * b) / p.W) % 4 == wi) blk[ng++] = b;
        } else {
          li0 = c ? li0_1 : li0_0;                // first block of this warp in chunk c
          ng = c ? ng_1 : ng_0;
        }
        const uint32_t tb = tmem + (uint32_t(32 * q) << 16) + uint32_t(slot * 256);
        if (!PERG && !masked && ng > 0) {
          const uint32_t te = bar_tempty(s, slot);
          const float* lse_c = lse2 + c * nn;
          if (ng == 4) p2_use<4>(tb, li0, lse_c, s22, te, lane, acc0, acc1);
          else if (ng == 3) p2_use<3>(tb, li0, lse_c, s22, te, lane, acc0, acc1);
          else if (ng == 2) p2_use<2>(tb, li0, lse_c, s22, te, lane, acc0, acc1);
          else p2_use<1>(tb, li0, lse_c, s22, te, lane, acc0, acc1);
          continue;
        }
        // General case: masked keys (the last tiles), blocks by query head (PERG).
        auto col = [&](int k) { return PERG ? blk[k] : li0 + 4 * k; };
        // Block k + 1 is loaded while block k is summed; the slot is released as soon as
        // the last block's load has landed.
        uint32_t v[2][16];
        if (ng > 0) {
          tmem_ld16(tb + uint32_t(col(0) * 16), v[0]);
          tmem_wait_ld(v[0]);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (k >= ng) break;
          if (k + 1 < ng) {
            tmem_ld16(tb + uint32_t(col(k + 1) * 16), v[(k + 1) & 1]);
          } else {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_tempty(s, slot));   // slot free: all of it loaded
          }
          uint32_t (&vk)[16] = v[k & 1];
          const int r0 = c * nn + col(k) * 16;
          if (masked) {                            // rows that cannot see key j drop out
#pragma unroll
            for (int e = 0; e < 16; ++e)
              if (j > (p.causal ? lim_base + (r0 + e) % p.W : lim_base)) vk[e] = 0xff800000u;
          }
          const float4* nl = reinterpret_cast<const float4*>(lse2 + r0);
          const bool second = PERG && (r0 / p.W) >= 4;     // head slot of this block
          uint64_t a0 = second ? acc2 : acc0, a1 = second ? acc3 : acc1;
#pragma unroll
          for (int e = 0; e < 16; e += 4) {
            const float4 b = nl[e >> 2];
            a0 = acc_exp2(a0, vk[e], vk[e + 1], s22, pk(b.x, b.y));
            a1 = acc_exp2(a1, vk[e + 2], vk[e + 3], s22, pk(b.z, b.w));
          }
          if (second) {
            acc2 = a0;
            acc3 = a1;
          } else {
            acc0 = a0;
            acc1 = a1;
          }
          if (k + 1 < ng) tmem_wait_ld(v[(k + 1) & 1]);
        }
        if (ng == 0) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar_tempty(s, slot));
        }
      }
      if (ok && j < p.L)
        raw_out[j] = PERG ? fmaxf(hsum(acc0, acc1), hsum(acc2, acc3)) : hsum(acc0, acc1);
    }
  }
  teardown(tmem);
}

// scores = max-pool over [j - radius, j + radius] (clipped to the row) of the sum of the
// four partial-sum planes (Section 3.3's pooling of the window scores).  One block per
// kPoolTile positions of one head: the plane sums of the tile and its halo are formed once
// in shared memory with coalesced loads, then every output takes its window maximum there.
constexpr int kPoolTile = 1024;
constexpr int kPoolThreads = 256;
constexpr int kMaxRadius = kMaxPoolRadius;

__global__ void __launch_bounds__(kPoolThreads)
maxpool_sum_kernel(const float* __restrict__ raw, float* __restrict__ out, int64_t L,
                   int64_t plane, int radius, int combine_max) {
  __shared__ float sum[kPoolTile + 2 * kMaxRadius];
  const int64_t tiles = ceil_div(L, kPoolTile);
  const int h = int(blockIdx.x / tiles);
  const int64_t base = (blockIdx.x % tiles) * kPoolTile;
  const float* r0 = raw + int64_t(h) * L;
  auto comb = [&](float a, float b, float c, float d) {
    return combine_max ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
  };
  auto at = [&](int64_t j) {                       // plane combination at position j
    return comb(__ldcg(r0 + j), __ldcg(r0 + plane + j), __ldcg(r0 + 2 * plane + j),
                __ldcg(r0 + 3 * plane + j));
  };
  // sum[i] holds position base - radius + i (-inf outside the row)
  const int span = kPoolTile + 2 * radius;
  // whole tile, rows a multiple of 4 positions long and 16-byte aligned buffers: one 16-byte
  // load per plane per thread (and one 16-byte store), the halo by scalar loads
  const bool vec = (L & 3) == 0 && base + kPoolTile <= L &&
                   ((reinterpret_cast<uintptr_t>(raw) | reinterpret_cast<uintptr_t>(out)) & 15) == 0;
  if (vec) {
    static_assert(kPoolTile == 4 * kPoolThreads, "four positions per thread");
    const int t = threadIdx.x;
    const int64_t j = base + 4 * t;
    const float4 a = __ldcg(reinterpret_cast<const float4*>(r0 + j));
    const float4 b = __ldcg(reinterpret_cast<const float4*>(r0 + plane + j));
    const float4 c = __ldcg(reinterpret_cast<const float4*>(r0 + 2 * plane + j));
    const float4 d = __ldcg(reinterpret_cast<const float4*>(r0 + 3 * plane + j));
    float* sp = sum + radius + 4 * t;
    sp[0] = comb(a.x, b.x, c.x, d.x);
    sp[1] = comb(a.y, b.y, c.y, d.y);
    sp[2] = comb(a.z, b.z, c.z, d.z);
    sp[3] = comb(a.w, b.w, c.w, d.w);
    if (t < 2 * radius) {
      const int i = t < radius ? t : kPoolTile + t;
      const int64_t jh = base - radius + i;
      sum[i] = jh >= 0 && jh < L ? at(jh) : -INFINITY;
    }
  } else {
    for (int i = threadIdx.x; i < span; i += kPoolThreads) {
      const int64_t jh = base - radius + i;
      sum[i] = jh >= 0 && jh < L ? at(jh) : -INFINITY;
    }
  }
  __syncthreads();
  float* o = out + int64_t(h) * L;
  if (vec) {
    const int i0 = 4 * threadIdx.x;
    float m[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) m[e] = sum[i0 + e + radius];
    for (int k = 0; k < 2 * radius + 1; ++k)
#pragma unroll
      for (int e = 0; e < 4; ++e) m[e] = fmaxf(m[e], sum[i0 + e + k]);
    *reinterpret_cast<float4*>(o + base + i0) = make_float4(m[0], m[1], m[2], m[3]);
  } else {
    for (int i = threadIdx.x; i < kPoolTile; i += kPoolThreads) {
      const int64_t j = base + i;
      if (j >= L) break;
      float m = sum[i + radius];
      for (int k = 0; k < 2 * radius + 1; ++k) m = fmaxf(m, sum[i + k]);
      o[j] = m;
    }
  }
}

// ---------------------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

// 2-D bf16 map over a [rows][128] row-major matrix, box {64 columns, box_rows}, 128B swizzle.
bool make_map(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cuuint64_t(kD), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(kD * 2)};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 148;
  return n;
}

}  // namespace

uint64_t g_score_wait_ns = 2000000000ull;
uint32_t g_score_flags = 0;

cudaError_t launch_passes(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                          int64_t L, int W, uint32_t flags, const float* head_weights,
                          const Ws& ws, cudaStream_t stream, unsigned passes) {
  TcParams p{};
  p.Hkv = Hkv;
  p.G = Hq / Hkv;
  p.W = W;
  p.GW = p.G * W;
  p.L = L;
  p.T = int(ceil_div(L, kTileKeys));
  const int nsm = sm_count();
  p.cph = nsm / Hkv;
  if (p.cph < 1) p.cph = 1;
  if (p.cph > p.T) p.cph = p.T;
  p.nrt = int(ceil_div(p.GW, 128));
  p.nparts = p.cph;
  if (p.nparts > kMaxScoreParts) return cudaErrorInvalidConfiguration;
  p.scale2 = kLog2e / sqrtf(float(kD));
  p.causal = (flags & SGDKV_SCORE_PROXY_QUERY) ? 0 : 1;
  p.agg = int((flags & SGDKV_SCORE_AGG_MASK) >> 1);
  p.head_w = head_weights;
  p.det = (flags & SGDKV_SCORE_DETERMINISTIC) ? 1 : 0;
  if (p.agg != 0 && !head_weights) return cudaErrorInvalidValue;
  if (p.agg == 1 && (W % 16 != 0 || W > 64 || p.G > 8)) return cudaErrorInvalidValue;
  p.wait_ns = g_score_wait_ns;
  p.flags = g_score_flags;

  CUtensorMap tm_q, tm_k;
  if (!make_map(&tm_q, q, uint64_t(Hq) * W, kQBoxRows) ||
      !make_map(&tm_k, K, uint64_t(Hkv) * L, kTileKeys))
    return cudaErrorInvalidValue;
  // K ring depth: as many 32 KB stages as fit next to each pass's other shared data.
  TcParams p1 = p, p2 = p;
  const size_t fixed1 = size_t(2) * p.nrt * 128 * 128 + kCtlBytes;   // Q padded to row tiles
  const size_t fixed2 = size_t(2) * p.GW * 128 + kCtlBytes + kMaxRows * sizeof(float);
  p1.nstages = int((kSmemLimit - fixed1) / kStageBytes);
  p2.nstages = int((kSmemLimit - fixed2) / kStageBytes);
  if (p1.nstages > kMaxStages) p1.nstages = kMaxStages;
  if (p2.nstages > kMaxStages) p2.nstages = kMaxStages;
  if (p1.nstages < 2 || p2.nstages < 2) return cudaErrorInvalidConfiguration;
  const size_t smem1 = fixed1 + size_t(p1.nstages) * kStageBytes;
  const size_t smem2 = fixed2 + size_t(p2.nstages) * kStageBytes;
  // the pass-1 row-merge buffer reuses the K ring once it is idle
  static_assert(4 * kMaxRows * sizeof(float2) <= size_t(2) * kStageBytes, "merge buffer");
  void (*pass1)(const CUtensorMap, const CUtensorMap, TcParams, Ws) =
      p.nrt == 1 ? score_pass1_tc<1>
                 : (p.nrt == 2 ? score_pass1_tc<2> : (p.nrt == 3 ? score_pass1_tc<3> : score_pass1_tc<4>));
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(pass1, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                int(smem1))) != cudaSuccess)
    return e;
  void (*pass2)(const CUtensorMap, const CUtensorMap, TcParams, Ws) =
      p.agg == 1 ? score_pass2_tc<true> : score_pass2_tc<false>;
  if ((e = cudaFuncSetAttribute(pass2, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                int(smem2))) != cudaSuccess)
    return e;
  const int grid = Hkv * p.cph;
  if (passes & 1u) {
    KernelTimer t(SGDKV_KERNEL_SCORE_PASS1, stream);
    pass1<<<grid, kThreads, smem1, stream>>>(tm_q, tm_k, p1, ws);
    note_launches(1);
  }
  if (passes & 2u) {
    KernelTimer t(SGDKV_KERNEL_SCORE_PASS2, stream);
    pass2<<<grid, kThreads, smem2, stream>>>(tm_q, tm_k, p2, ws);
    note_launches(1);
  }
  return cudaGetLastError();
}

cudaError_t launch_score_raw(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                             int64_t L, int W, uint32_t flags, const float* head_weights,
                             const Ws& ws, cudaStream_t stream) {
  return launch_passes(q, K, Hq, Hkv, L, W, flags, head_weights, ws, stream, 3u);
}

cudaError_t launch_pool(const Ws& ws, int Hkv, int64_t L, int pool, uint32_t flags,
                        float* scores_out, cudaStream_t stream) {
  if (pool < 1 || pool / 2 > kMaxRadius) return cudaErrorInvalidValue;
  {
    KernelTimer t(SGDKV_KERNEL_POOL, stream);
    const unsigned blocks = unsigned(int64_t(Hkv) * ceil_div(L, kPoolTile));
    const bool combine_max = (flags & SGDKV_SCORE_AGG_MASK) == SGDKV_SCORE_AGG_IPT_MAX;
    maxpool_sum_kernel<<<blocks, kPoolThreads, 0, stream>>>(ws.raw, scores_out, L,
                                                            int64_t(Hkv) * L, pool / 2,
                                                            combine_max ? 1 : 0);
  }
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_score(const __nv_bfloat16* q, const __nv_bfloat16* K, int Hq, int Hkv,
                         int64_t L, int W, int pool, uint32_t flags, const float* head_weights,
                         float* scores_out, const Ws& ws, cudaStream_t stream) {
  if (pool < 1 || pool / 2 > kMaxRadius) return cudaErrorInvalidValue;
  cudaError_t e = launch_score_raw(q, K, Hq, Hkv, L, W, flags, head_weights, ws, stream);
  if (e != cudaSuccess) return e;
  return launch_pool(ws, Hkv, L, pool, flags, scores_out, stream);
}

}  // namespace sgdkv
