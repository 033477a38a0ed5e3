/*
 * sgdkv.h: C-ABI of libsgdkv, the GB300 (sm_103a) implementation of the SGD-KV
 * inference-time KV-cache compression step ("Summarization Guided KV Cache Compression").
 *
 * Per layer, after prefill, the step
 *   1. scores every cached token of each KV head with the last W window queries
 *      (causal softmax of q.k/sqrt(d), summed over the window and the GQA group),
 *   2. smooths the scores with a 1-D max-pool,
 *   3. keeps each head's b_h best tokens (sink and recent tokens always kept), where b_h
 *      comes from the summarization-score budget allocation of Section 3.3 / Algorithm 1,
 *   4. gathers the kept K/V rows into a flat per-head variable-length cache.
 *
 * Conventions shared by every entry point:
 *   - The caller owns all memory.  The library allocates nothing and keeps no pointer past
 *     a call.  Device buffers are plain device pointers (cudaMalloc or torch storage).
 *   - bf16 tensors are passed as `const void*` to raw bfloat16 storage, row-major:
 *       q_win [Hq][W][d]     window queries, query head q belongs to KV head q / (Hq/Hkv)
 *       K, V  [Hkv][L][d]    one layer's prefilled cache
 *     Every device pointer must be 16-byte aligned.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).  Device
 *     work is enqueued asynchronously on it; host-side argument checks happen before any
 *     launch and leave all outputs untouched on error.
 *   - `workspace` is a device buffer of at least sgdkv_workspace_bytes(...) bytes, 256-byte
 *     aligned, zero-filled once by the caller before its first use (its first word is the
 *     device status word; it also holds the scorer's key-tile counters, which every call
 *     leaves at zero).  Calls that share a workspace must be ordered (same stream or
 *     synchronised); calls with separate workspaces may run concurrently.
 *   - Device-side failures (a bounded wait that ran out) are recorded in a status word in
 *     the workspace and reported by sgdkv_last_error.  No call aborts the process, traps,
 *     or falls back to the CPU.
 *   - v1 limits: d == 128; Hq % Hkv == 0; G*W a multiple of 32 and <= 512 (G = Hq/Hkv);
 *     Hkv <= SGDKV_MAX_KV_HEADS; Hkv*L < 2^31; pool odd in [1, 63].
 */
#ifndef SGDKV_H_
#define SGDKV_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SGDKV_API __attribute__((visibility("default")))
#else
#define SGDKV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define SGDKV_MAX_KV_HEADS 64
#define SGDKV_HEAD_DIM 128

typedef enum {
  SGDKV_OK = 0,
  SGDKV_ERR_INVALID_ARG = 1,       /* null pointer, bad shape, misaligned pointer        */
  SGDKV_ERR_INFEASIBLE_BUDGET = 2, /* total budget outside [N*floor, N*context_len]      */
  SGDKV_ERR_WORKSPACE = 3,         /* workspace missing, too small or misaligned         */
  SGDKV_ERR_CUDA = 4,              /* a CUDA runtime call or launch failed               */
  SGDKV_ERR_TIMEOUT = 5,           /* a device-side bounded wait ran out                 */
  SGDKV_ERR_UNSUPPORTED = 6,       /* shape outside the v1 limits above                  */
  SGDKV_ERR_INTERNAL = 7           /* a device-side consistency check failed; the access */
                                   /* it guarded was skipped                             */
} sgdkv_status;

/* Allocation modes of sgdkv_allocate_budgets. */
#define SGDKV_ALLOC_GREEDY 0       /* Algorithm 1, excess to top-scoring heads in turn     */
#define SGDKV_ALLOC_PROPORTIONAL 1 /* water level: min(cap, lambda * S_h)                  */
#define SGDKV_ALLOC_THRESHOLD 2    /* appendix "thr": scores below the mean zeroed, greedy */
#define SGDKV_ALLOC_REVERSE 3      /* appendix "Reverse": greedy, every middle share inverted */

/* Static description of a status code. Never NULL. */
SGDKV_API const char* sgdkv_status_string(int status);

/* Library version, major*10000 + minor*100 + patch. */
SGDKV_API int sgdkv_version(void);

/*
 * Head-level budget allocation (host only, deterministic, no device work).
 * Follows Section 3.3, Eq. (2) and Appendix A.1, Algorithm 1 of the paper.
 *
 * head_scores  [n_heads] host floats, one summarization score per (layer, KV head); the
 *              allocation runs jointly over all of them.  Finite, >= 0; all zero means
 *              uniform.
 * context_len  C, tokens per head before compression.
 * total_budget T, kept tokens summed over all heads, floors included.
 * floor        f = b_sink + b_window, kept by every head; the middle share is capped at
 *              M = C - f.
 * mode         SGDKV_ALLOC_*.
 * budgets_out  [n_heads] host int64: f <= b_h <= C and sum b_h == T exactly.
 *
 * The middle pool P = T - n_heads*f is shared in proportion to S_h = s_h / sum(s)
 * (Eq. 2), shares above M are capped and their excess redistributed (Algorithm 1), and
 * the real shares are rounded by largest remainder (ties: higher S_h, then lower index).
 * SGDKV_ALLOC_REVERSE (the "SGD-KV (Reverse)" row of the appendix's ablation, Table 3):
 * the greedy allocation of T, then every head's middle share m_h = b_h - f becomes M - m_h
 * (a head given 10 % keeps 90 %), so for this mode sum b_h == n*(C + f) - T instead.
 * All arithmetic is IEEE double in a fixed order, so results are bit-reproducible.
 * Errors: INVALID_ARG (null, n_heads <= 0, f outside [0, C], bad mode, negative/NaN/Inf
 * score), INFEASIBLE_BUDGET (T outside [n*f, n*C]).  budgets_out untouched on error.
 */
SGDKV_API sgdkv_status sgdkv_allocate_budgets(const float* head_scores, int32_t n_heads,
                                    int64_t context_len, int64_t total_budget, int64_t floor,
                                    int32_t mode, int64_t* budgets_out);

/*
 * Head scores of the "SGD-KV + HeadKV" row of the appendix's ablation (Table 3): two score
 * sets over the same heads (summarization scores and HeadKV's retrieval-reasoning scores),
 * each normalised to sum one (an all-zero set counts as uniform), then averaged:
 *   scores_out[h] = (a[h] / sum(a) + b[h] / sum(b)) / 2
 * with the sums taken in ascending head order in IEEE double and the result rounded once
 * to float.  The output is a head_scores input of sgdkv_allocate_budgets.  Host only.
 * a, b, scores_out  [n_heads] host floats (scores_out may alias a or b).
 * Errors: INVALID_ARG (null, n_heads <= 0, negative/NaN/Inf score); scores_out untouched.
 */
SGDKV_API sgdkv_status sgdkv_mix_head_scores(const float* a, const float* b, int32_t n_heads,
                                             float* scores_out);

/* Workspace bytes needed by sgdkv_score / sgdkv_compact / sgdkv_compress_layer for this
 * shape (one size serves all three).  Returns 0 for shapes outside the v1 limits. */
SGDKV_API size_t sgdkv_workspace_bytes(int32_t Hq, int32_t Hkv, int64_t L, int32_t d, int32_t W);

/*
 * Window scoring (Section 3.3 and Section 5: cumulative attention of the final
 * observation window, SnapKV-style), followed by max-pooling.
 *
 *   raw[h][j]    = sum_{g<G} sum_{w<W} softmax_j( q[h*G+g][w] . K[h][j] / sqrt(d) )
 *                  where window query w sits at position L-W+w and sees keys j <= L-W+w;
 *   scores[h][j] = max of raw[h][t] over t in [j - pool/2, j + pool/2] within [0, L).
 *
 * q_win      device bf16 [Hq][W][d];  K  device bf16 [Hkv][L][d]
 * pool       odd kernel size; 1 returns the raw scores.
 * scores_out device fp32 [Hkv][L].
 * Reproducibility: the scoring CTAs claim key tiles dynamically, and how each window row's
 * softmax denominator is summed follows the claims, so two calls on the same input agree to
 * within fp32 rounding (relative ~1e-6), not bit for bit (sgdkv_score_ex with
 * SGDKV_SCORE_DETERMINISTIC: bit for bit).
 * Errors: INVALID_ARG, UNSUPPORTED, WORKSPACE, CUDA (launch failure).
 */
SGDKV_API sgdkv_status sgdkv_score(const void* q_win, const void* K, int32_t Hq, int32_t Hkv, int64_t L,
                         int32_t d, int32_t W, int32_t pool, float* scores_out,
                         void* workspace, size_t ws_bytes, void* stream);

/*
 * sgdkv_score with scoring flags.  flags == 0 (and head_weights NULL) is sgdkv_score.
 *
 * SGDKV_SCORE_PROXY_QUERY: the W rows of q_win per query head are an external query (the
 * proxy-query setting of the paper's query ablation, Section "Ablation Study: Impact of
 * Query on Token Selection", Table 3: a fixed task-agnostic prompt stands in for the
 * unknown question).  Such queries come after the whole context, so every row sees all L
 * keys: no causal mask.  (The query-unaware setting of the same ablation is ordinary
 * scoring of a context that ends before the question: flags without this bit, that L.)
 *
 * Aggregation over the GQA group (flag bits 1-2; the appendix's head configuration
 * variants, "Ipt." rows of its ablation table).  With A_g[j] the cumulative window
 * attention of query head g of the group (sum over its W rows of the softmax) and w_g its
 * summarization score, head_weights[q] = w of query head q:
 *   SGDKV_SCORE_AGG_SUM      (0)  raw[j] = sum_g A_g[j]            (sgdkv_score)
 *   SGDKV_SCORE_AGG_IPT_MAX       raw[j] = max_g w_g A_g[j]        ("Ipt., Max")
 *   SGDKV_SCORE_AGG_IPT_MEAN      raw[j] = mean_g w_g A_g[j]       ("Ipt., Mean")
 *   SGDKV_SCORE_AGG_IPT_ONLY      raw[j] = A_g*[j], g* the group's highest w (lower g on
 *                                 ties)                            ("Ipt., Only")
 * then max-pooling as in sgdkv_score.  head_weights: device fp32 [Hq], finite and >= 0
 * (required for the IPT modes, ignored otherwise); a negative or non-finite weight is
 * found on the device, records SGDKV_ERR_INVALID_ARG in the workspace status word
 * (sgdkv_last_error) and its head contributes nothing.  SGDKV_SCORE_AGG_IPT_MAX needs
 * W in {16, 32, 48, 64} and G <= 8 (UNSUPPORTED otherwise).
 * SGDKV_SCORE_DETERMINISTIC (bit 3): bit-reproducible scores.  By default the scoring CTAs
 * of a KV head claim its key tiles dynamically (the CTAs that start late, while other
 * kernels hold SMs, take fewer), so each window row's softmax denominator is summed in an
 * order that varies between calls.  With this bit the first pass gives CTA c of a head the
 * key tiles c, c + C, c + 2C, ... (C CTAs per head), and every sum of both passes follows a
 * fixed order: two calls on the same input and device give the same scores bit for bit,
 * whatever else the GPU runs meanwhile.  The price is load balance: a CTA that starts late
 * still has its whole share of tiles.
 * Unknown flag bits, or an IPT mode without head_weights: INVALID_ARG.  Other arguments and
 * errors as sgdkv_score.
 */
#define SGDKV_SCORE_PROXY_QUERY 1u
#define SGDKV_SCORE_AGG_SUM (0u << 1)
#define SGDKV_SCORE_AGG_IPT_MAX (1u << 1)
#define SGDKV_SCORE_AGG_IPT_MEAN (2u << 1)
#define SGDKV_SCORE_AGG_IPT_ONLY (3u << 1)
#define SGDKV_SCORE_AGG_MASK (3u << 1)
#define SGDKV_SCORE_DETERMINISTIC (1u << 3)
SGDKV_API sgdkv_status sgdkv_score_ex(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                                      int64_t L, int32_t d, int32_t W, int32_t pool,
                                      uint32_t flags, const float* head_weights,
                                      float* scores_out, void* workspace, size_t ws_bytes,
                                      void* stream);

/*
 * The two halves of sgdkv_score_ex, for callers that max-pool on another stream (the
 * benchmark overlaps layer l's pooling and compaction with layer l+1's scoring).
 * sgdkv_score_raw runs both scoring passes and leaves raw[h][j] (the window scores before
 * pooling, of sgdkv_score / sgdkv_score_ex with these flags) in the workspace as partial
 * sums; sgdkv_pool_raw max-pools them into scores_out.  In between the workspace holds the
 * raw scores: any other call on it, sgdkv_score_raw of the next layer included, overwrites
 * them, so a caller that overlaps layers alternates two workspaces.  sgdkv_pool_raw must
 * get the Hkv, L and flags the raw scores were made with (the aggregation bits choose how
 * the partial sums combine).  Arguments and errors as sgdkv_score_ex; the workspace is the
 * one sized by sgdkv_workspace_bytes.
 */
SGDKV_API sgdkv_status sgdkv_score_raw(const void* q_win, const void* K, int32_t Hq, int32_t Hkv,
                                       int64_t L, int32_t d, int32_t W, uint32_t flags,
                                       const float* head_weights, void* workspace,
                                       size_t ws_bytes, void* stream);
SGDKV_API sgdkv_status sgdkv_pool_raw(const void* workspace, size_t ws_bytes, int32_t Hkv,
                                      int64_t L, int32_t pool, uint32_t flags, float* scores_out,
                                      void* stream);

/*
 * sgdkv_score_raw's two passes as separate calls (steps a2 and a3 of the scoring: Section
 * 3.3's softmax over the keys needs every window row's normaliser before any key's sum).
 * sgdkv_window_stats: window logits t_rj = q_r . k_j / sqrt(d) and, per window row r, the
 * online (max, sum of exp) over the keys the row sees, kept in the workspace.
 * sgdkv_window_sums: recomputes the logits and sums exp(t_rj - lse_r) over the window rows
 * (and the GQA group, with the flags' aggregation) per key, from the statistics a
 * sgdkv_window_stats call with the same arguments left in the same workspace; the raw
 * scores then wait there for sgdkv_pool_raw.  The workspace holds the statistics in
 * between: a caller that overlaps layers (one layer's sums beside the next layer's
 * statistics) gives each layer in flight its own workspace.  Arguments and errors as
 * sgdkv_score_raw.
 */
SGDKV_API sgdkv_status sgdkv_window_stats(const void* q_win, const void* K, int32_t Hq,
                                          int32_t Hkv, int64_t L, int32_t d, int32_t W,
                                          uint32_t flags, const float* head_weights,
                                          void* workspace, size_t ws_bytes, void* stream);
SGDKV_API sgdkv_status sgdkv_window_sums(const void* q_win, const void* K, int32_t Hq,
                                         int32_t Hkv, int64_t L, int32_t d, int32_t W,
                                         uint32_t flags, const float* head_weights,
                                         void* workspace, size_t ws_bytes, void* stream);

/*
 * sgdkv_score without a workspace argument, for callers that cannot allocate device
 * memory (for example code running where the allocator is owned by someone else, or a
 * plugin that may only receive tensors).  No counterpart in the paper: the computation
 * and the results are those of sgdkv_score with pool, scores_out as there.
 *
 * The scratch is a static 64 MiB device array inside this library, held on every GPU that
 * loads it until the process exits.  Shapes needing more than that (the status word, the
 * per-CTA row statistics and the four raw-score planes, about 1.3 MiB * Hkv + 16 * Hkv * L
 * bytes) are rejected with SGDKV_ERR_WORKSPACE before any device work.  The call allocates
 * nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * status_out: optional device pointer to one uint32; receives the device-side status of
 *             this call (SGDKV_OK or SGDKV_ERR_TIMEOUT / SGDKV_ERR_INTERNAL), as
 *             sgdkv_last_error would report it.  NULL skips the copy.
 * All calls on a device share the one scratch array, which keeps the last call's
 * contents; the status word and the tile counters are cleared at the start of every call.
 * Calls that can overlap on the GPU (different streams, no ordering between them) race on
 * it and give undefined results.  The first call on each device looks the scratch up (cudaGetSymbolAddress)
 * with that device current; make that first call before any stream capture.
 */
SGDKV_API sgdkv_status sgdkv_score_static(const void* q_win, const void* K, int32_t Hq,
                                          int32_t Hkv, int64_t L, int32_t d, int32_t W,
                                          int32_t pool, float* scores_out, uint32_t* status_out,
                                          void* stream);

/*
 * Token selection and gather (Section 3.3): per KV head keep positions [0, n_sink) and
 * [L - n_recent, L), plus the (b_h - n_sink - n_recent) middle positions with the highest
 * scores (equal scores: lower position first).  Kept positions are written ascending.
 *
 * K, V            bf16 [Hkv][L][d]: device memory, or pinned host memory that the device
 *                 addresses directly (cudaHostAlloc, cudaHostRegister).  Only the kept rows
 *                 are read (by the gather), so a cache held in host memory crosses the host
 *                 link for the kept rows alone.
 * scores          device fp32 [Hkv][L], finite and >= 0 (as produced by sgdkv_score); -0.0
 *                 counts as +0.0.  NaN or negative scores are outside the contract: the
 *                 selection is then unspecified, though every write stays in bounds
 * budgets         HOST int64 [Hkv], n_sink + n_recent <= b_h <= L
 * indices_out     device int32 [sum b_h]: kept positions, head by head
 * cu_seqlens_out  device int32 [Hkv + 1]: cu[0] = 0, cu[h+1] = cu[h] + b_h
 * K_out, V_out    device bf16 [sum b_h][d]: row cu[h]+i = K[h][indices_out[cu[h]+i]]
 * Errors: INVALID_ARG, UNSUPPORTED, WORKSPACE, CUDA.
 */
SGDKV_API sgdkv_status sgdkv_compact(const void* K, const void* V, const float* scores,
                           const int64_t* budgets, int32_t Hkv, int64_t L, int32_t d,
                           int64_t n_sink, int64_t n_recent, int32_t* indices_out,
                           int32_t* cu_seqlens_out, void* K_out, void* V_out, void* workspace,
                           size_t ws_bytes, void* stream);

/*
 * sgdkv_pool_raw followed by sgdkv_compact in one call (Section 3.3: max-pool of the window
 * scores, then the selection and gather), reading the raw scores that sgdkv_score_raw or
 * sgdkv_window_sums left in score_workspace.  Where the selection keeps each slice of a row
 * in registers (rows up to 524288 positions on a GPU with 16-CTA clusters), the selection
 * kernel pools its own slice and no pool kernel is launched; longer rows take the two
 * kernels.  Either way scores_out receives the pooled scores bit for bit as sgdkv_pool_raw
 * writes them, and the kept positions and rows are those sgdkv_compact gives on them.
 *
 * score_workspace, score_ws_bytes  the workspace holding the raw scores (read only); pool and
 *                 flags as given to sgdkv_pool_raw (the Hkv, L and flags of the scoring call)
 * scores_out      device fp32 [Hkv][L], 16-byte aligned (required)
 * workspace       the compaction's own workspace (device-side errors are recorded there);
 *                 may be score_workspace itself
 * Other arguments as sgdkv_compact.  A caller that overlaps layers may start the next
 * scoring call on score_workspace only after this call.  Errors: INVALID_ARG, UNSUPPORTED,
 * WORKSPACE, CUDA.
 */
SGDKV_API sgdkv_status sgdkv_pool_compact(const void* score_workspace, size_t score_ws_bytes,
                                          int32_t pool, uint32_t flags, const void* K,
                                          const void* V, const int64_t* budgets, int32_t Hkv,
                                          int64_t L, int32_t d, int64_t n_sink,
                                          int64_t n_recent, float* scores_out,
                                          int32_t* indices_out, int32_t* cu_seqlens_out,
                                          void* K_out, void* V_out, void* workspace,
                                          size_t ws_bytes, void* stream);

/*
 * Decode attention over the compressed cache (what generation computes with it: Section
 * 3.3, the kept tokens are each head's history; Appendix, Configuration, the cache is kept
 * per KV head before the values are repeated for the query heads of a GQA group): for every
 * query head qh and new token t,
 *   out[qh][t] = sum_i softmax_i(q[qh][t] . K_cache[c + i] / sqrt(d)) V_cache[c + i],
 * i over the b_h kept rows of KV head h = qh / G, c = b_0 + ... + b_{h-1} (the layout
 * sgdkv_compact writes: pass the budgets it was given).  A head with b_h = 0 gives zeros.
 *
 * q         device bf16 [Hq][n_tok][d], 16-byte aligned; G * n_tok <= 16 (UNSUPPORTED
 *           otherwise; G = Hq / Hkv)
 * K_cache,
 * V_cache   device bf16 [sum b_h][d], 16-byte aligned (may be NULL when every b_h is 0)
 * budgets   HOST int64 [Hkv], b_h >= 0, sum < 2^31
 * out       device fp32 [Hq][n_tok][d], 16-byte aligned
 * workspace device, 256-byte aligned, sgdkv_decode_workspace_bytes(Hq, Hkv, n_tok, d,
 *           sum b_h) bytes (0 there: shape unsupported); the per-warp partials.  The size
 *           grows with sum b_h up to a bound (1.3 MB at Hkv = 4), so a workspace sized for
 *           the largest cache serves every smaller one
 * Arithmetic: logits with bf16 products and fp32 sums, softmax in fp32 (log2 units), the
 * weights rounded to bf16 for the value sum, normalised by the sum of the rounded weights;
 * the output is a convex combination of the head's value rows, within 2^-8 max|v| of the
 * exact one.  Asynchronous on stream.  Two kernels, both launched as programmatic dependents
 * of what precedes them on the stream: a call placed right after another decode call (one
 * per layer, say) starts streaming its cache while the previous call's merge runs, so its
 * q, K_cache, V_cache and budgets-derived layout must not be outputs of that previous call
 * (out of one call is never an input of the next in a decode step); it rewrites the shared
 * workspace only after the previous call has completed.  Errors: INVALID_ARG, UNSUPPORTED,
 * WORKSPACE, CUDA.
 */
SGDKV_API size_t sgdkv_decode_workspace_bytes(int32_t Hq, int32_t Hkv, int32_t n_tok, int32_t d,
                                              int64_t total_rows);
SGDKV_API sgdkv_status sgdkv_decode_attention(const void* q, int32_t Hq, int32_t Hkv,
                                              int32_t n_tok, int32_t d, const void* K_cache,
                                              const void* V_cache, const int64_t* budgets,
                                              float* out, void* workspace, size_t ws_bytes,
                                              void* stream);

/*
 * The whole per-layer step: sgdkv_score followed by sgdkv_compact on the same stream,
 * keeping the pooled scores in the workspace.  scores_out may be NULL; when given, it
 * receives the pooled scores as sgdkv_score would.  K must be device memory (the scorer
 * streams it with TMA); V may be pinned host memory as in sgdkv_compact.  Other arguments
 * as above.
 */
SGDKV_API sgdkv_status sgdkv_compress_layer(const void* q_win, const void* K, const void* V,
                                  const int64_t* budgets, int32_t Hq, int32_t Hkv, int64_t L,
                                  int32_t d, int32_t W, int32_t pool, int64_t n_sink,
                                  int64_t n_recent, float* scores_out, int32_t* indices_out,
                                  int32_t* cu_seqlens_out, void* K_out, void* V_out,
                                  void* workspace, size_t ws_bytes, void* stream);

/*
 * Diagnostics: number of kernel launches this process has issued through libsgdkv so far
 * (all entry points, all devices).  A launch issued into a stream that is being captured
 * into a CUDA graph counts once, at capture.  No counterpart in the paper; used to report how
 * many of the library's kernels a timed region ran.
 */
SGDKV_API uint64_t sgdkv_launch_count(void);

/*
 * Diagnostics: text of the last CUDA runtime error this library saw on the calling thread
 * ("no error" if none).  Explains an SGDKV_ERR_CUDA result.  Never NULL.
 */
SGDKV_API const char* sgdkv_last_cuda_error_string(void);

/*
 * Diagnostics: per-kernel timing.  While bit k of kind_mask is set, every kernel of kind k
 * the library launches is bracketed by CUDA events on its launch stream (mask 0 turns timing
 * off; each bracket adds two event records to the stream).  sgdkv_debug_kernel_timing synchronises
 * the recorded events of one kernel kind, returns their summed duration in milliseconds and
 * their count, and forgets them.  A launch issued while its stream is being captured into a
 * CUDA graph is bracketed by event-record nodes of that graph: its record is read after the
 * graph has been launched (the last launch of the graph), and a graph that has not been
 * launched yet makes the call fail with CUDA.  No counterpart in the paper; used by the
 * benchmark to time its dominant kernel inside the timed region.  Errors: INVALID_ARG, CUDA.
 */
#define SGDKV_KERNEL_SCORE_PASS1 0   /* window logits, per-row max and sum  */
#define SGDKV_KERNEL_SCORE_PASS2 1   /* per-key sum of normalised weights   */
#define SGDKV_KERNEL_POOL 2          /* max-pool of the raw scores          */
#define SGDKV_KERNEL_SELECT 3        /* threshold select and ordered compaction */
#define SGDKV_KERNEL_GATHER 4        /* K/V row copy                        */
#define SGDKV_KERNEL_DECODE 5        /* decode attention (partials, merge)  */
#define SGDKV_KERNEL_KINDS 6
SGDKV_API void sgdkv_debug_enable_kernel_timing(uint32_t kind_mask);
SGDKV_API sgdkv_status sgdkv_debug_kernel_timing(int kind, double* total_ms, int64_t* launches);

/*
 * Test hook (no counterpart in the paper): sets the time bound, in nanoseconds, of every
 * device-side wait in the scoring kernels (0 restores the default of 2 s), and flags:
 * bit 0 makes the scoring kernels' MMA issuer first wait on a barrier nothing signals, so
 * that the wait runs out, SGDKV_ERR_TIMEOUT is recorded and the kernels drain and exit.
 * Process-wide; affects launches issued after the call.  Not thread-safe.
 */
SGDKV_API void sgdkv_debug_set_score_hooks(uint32_t flags, uint64_t wait_ns);

/*
 * Synchronises `stream`, then returns and clears the first device-side failure recorded
 * in `workspace` since the last call (SGDKV_OK if none), or SGDKV_ERR_CUDA if the stream
 * itself reports an error.
 */
SGDKV_API sgdkv_status sgdkv_last_error(void* workspace, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SGDKV_H_ */
