/*
 * kv_evict.h -- C ABI of the GB300 (sm_103a) diversified KV-eviction step.
 *
 * The step is the end-of-prefill token eviction of "Beyond Mean Attention:
 * Diversity-Aware, Layer-Wise Scoring for KV Cache Eviction" (Section 3). For every
 * (request, layer, KV head) -- a "unit" -- it
 *   1. scores every prefix token i by the attention A[q][i] it receives from the
 *      observation window, the last W query positions (Section 3.1, Eq. 1);
 *   2. reduces those scores over the window rows to the mean mu_i (Eq. 1) and the
 *      sample standard deviation sigma_i (Eq. 3);
 *   3. max-pools mu and sigma over the candidate tokens (Section 3.1 keeps the
 *      baselines' max-pooling), forms the base score s_i = mu_i + lambda1 * sigma_i
 *      (Eq. 2 without the redundancy term), restricts the candidates to the top
 *      4B tokens by s (Section 3.2), normalises s by its maximum (Eq. 5) and admits
 *      B tokens greedily by s~_i + lambda2 * corr(i, S) (Eq. 4, Eq. 5);
 *   4. gathers the kept key/value rows into a compact cache.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  * Symbols: N_L layers, Hq query heads, Hkv KV heads, G = Hq / Hkv (GQA group),
 *    d = head_dim, W = window, B = budget, n_req requests with prefix lengths L_r,
 *    SL = sum_r L_r, Lc_r = L_r - W candidate tokens of request r.
 *  * The window rows of unit (r, l, h) are the G query heads h*G .. h*G+G-1, each
 *    with its W window queries: n = G*W rows, row index g*W + w, at token position
 *    L_r - W + w. Causal masking: that row attends to keys 0 .. L_r - W + w.
 *  * All tensors are row-major, in device memory, allocated and owned by the
 *    caller; all but k and v are dense. bf16 tensors are passed as uint16_t bit
 *    patterns.
 *      q_win  [N_L][n_req][Hq][W][d]      bf16  window queries (after RoPE)
 *      k, v   [N_L][Hkv][SL][d]           bf16  prefix keys/values (after RoPE);
 *                                               request r occupies tokens
 *                                               off_r .. off_r + L_r - 1,
 *                                               off_r = L_0 + ... + L_{r-1}.
 *                                               Dense by default; any other
 *                                               strides between layers, heads and
 *                                               tokens through
 *                                               kv_evict_plan_set_kv_strides
 *      mu, sigma  packed per request: request r holds [N_L][Hkv][L_r] fp32 at
 *                 element offset N_L*Hkv*off_r
 *      indices    [n_req][N_L][Hkv][B] int32, kept candidate positions in
 *                 ascending order, -1 after the first min(B_l, Lc_r) entries
 *                 (B_l = B unless the plan has per-layer budgets, see
 *                 kv_evict_plan_layered)
 *      order      [n_req][N_L][Hkv][B] int32, the same positions in admission
 *                 order (optional)
 *      margins    [n_req][N_L][Hkv][B] fp32, per admission the gap between the
 *                 best and the second-best greedy value (optional)
 *      k_out, v_out [n_req][N_L][Hkv][B+W][d] bf16: rows 0 .. m-1 are the kept
 *                 candidates in ascending position (m = min(B_l, Lc_r)), rows
 *                 m .. m+W-1 the W window tokens, remaining rows zero.
 *  * Every pointer must be 16-byte aligned; q_win and k additionally 128-byte.
 *  * stream is a cudaStream_t passed as void*. Every device call is
 *    asynchronous on that stream and returns after the launches; device-side
 *    failures (a bounded wait that ran out) are reported by kv_evict_status.
 *  * Host validation failures return before any launch and write nothing.
 *  * A plan is immutable after kv_evict_plan and may be used from several host
 *    threads; a workspace must not be shared by calls that overlap on the GPU.
 */
#ifndef KV_EVICT_H
#define KV_EVICT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KVE_OK = 0,
  KVE_EINVAL = 1,   /* invalid argument or unsupported shape (host check)     */
  KVE_ECUDA = 2,    /* a CUDA runtime/driver call failed                      */
  KVE_ETIMEOUT = 3, /* a device-side bounded wait ran out (kv_evict_status)   */
  KVE_ENOMEM = 4    /* host allocation failed                                 */
} kve_status;

typedef struct {
  int32_t num_layers;       /* N_L >= 1                                        */
  int32_t num_q_heads;      /* Hq, a multiple of num_kv_heads                  */
  int32_t num_kv_heads;     /* Hkv >= 1                                        */
  int32_t head_dim;         /* d; this build supports d = 128                  */
  int32_t window;           /* W >= 1, with G*W <= 128                         */
  int32_t budget;           /* B >= 1 kept candidates per unit (the window is
                               kept in addition)                               */
  int32_t pool_kernel;      /* odd k, 1 <= k <= 255; max-pool of mu and sigma,
                               stride 1, window clipped to [0, Lc); 1 = none    */
  int32_t candidate_factor; /* greedy pool C = min(factor*B, Lc); Section 3.2
                               uses 4; 0 = every candidate                     */
  float norm_eps;           /* positive clamp of max_j s_j in Eq. 5            */
} kve_config;

typedef struct kve_plan kve_plan;

/* Validate cfg and the host array seq_lens[n_req] (every L_r > W), and build the
 * host-side schedule. *workspace_bytes receives the size of the device workspace
 * that kv_evict_score and kv_evict_select need (caller-allocated, 256-byte
 * aligned). The plan owns host memory only. Section 3 defines the shapes. */
kve_status kv_evict_plan(const kve_config* cfg, const int64_t* seq_lens,
                         int32_t n_req, kve_plan** plan_out,
                         size_t* workspace_bytes);

/* kv_evict_plan with a budget per layer: layer_budgets is a HOST array [N_L] with
 * 1 <= B_l <= cfg->budget; layer l keeps min(B_l, Lc_r) candidates (candidate pool
 * min(factor * B_l, Lc_r)). cfg->budget stays the row stride of indices, order,
 * margins (B) and of the compact cache (B + W). PyramidKV (Section 3.1) decreases
 * the budget with depth while keeping the total of the uniform allocation; see
 * kv_evict_budget_pyramid. layer_budgets = NULL is kv_evict_plan. */
kve_status kv_evict_plan_layered(const kve_config* cfg, const int64_t* seq_lens,
                                 int32_t n_req, const int32_t* layer_budgets,
                                 kve_plan** plan_out, size_t* workspace_bytes);

/* Flags of kv_evict_plan_ex. */
#define KVE_PLAN_PER_QUERY_HEAD 1

/* kv_evict_plan_layered with flags (0 = kv_evict_plan_layered).
 * KVE_PLAN_PER_QUERY_HEAD: every query head selects its own tokens. The paper leaves
 * the GQA grouping open; the default pools the G*W window rows of the query heads
 * that share a KV head into one unit (n = G*W rows, one selection per KV head).
 * With this flag a unit is (request, layer, query head): its n = W rows are that
 * head's window queries, its keys those of its KV head (query head hq reads KV head
 * hq / G), and the selection, the compact cache and every per-unit array are
 * indexed by query head: mu, sigma [n_req][N_L][Hq][L_r]; indices, order, margins
 * [n_req][N_L][Hq][B]; k_out, v_out [n_req][N_L][Hq][B+W][d]. Inputs keep their
 * layouts. Other flag bits: KVE_EINVAL. */
kve_status kv_evict_plan_ex(const kve_config* cfg, const int64_t* seq_lens,
                            int32_t n_req, const int32_t* layer_budgets,
                            int32_t flags, kve_plan** plan_out,
                            size_t* workspace_bytes);

void kv_evict_plan_destroy(kve_plan* plan);

/* Layout of k and v for later calls with this plan, so that a serving engine's cache
 * is read in place: strides[3] = element strides between layers, KV heads and
 * tokens (in that order) of the prefix keys (k_strides) and values (v_strides);
 * element (layer l, KV head h, token t, dim j) sits at l*s[0] + h*s[1] + t*s[2] + j,
 * with t = off_r + i for key i of request r (off_r as above). A row of d elements
 * stays contiguous. NULL is the dense default {Hkv*SL*d, SL*d, d}; a token-major
 * cache [N_L][SL][Hkv][d] is {SL*Hkv*d, d, Hkv*d}. Every stride must be a multiple
 * of 8 elements (16 bytes) and below 2^37, and the token stride at least d;
 * otherwise KVE_EINVAL and the plan is unchanged. Call it before the plan is used
 * on any stream; it changes the plan (not thread-safe with calls that use it). */
kve_status kv_evict_plan_set_kv_strides(kve_plan* plan, const int64_t* k_strides,
                                        const int64_t* v_strides);

/* Test hook: limit (ns) of every device-side bounded wait of later calls with this
 * plan (default 2e9), and a fault to inject on the host-chosen unit 0:
 * fault = 1 makes its row statistics never publish, so its column pass waits
 * out the limit and kv_evict_status reports KVE_ETIMEOUT. fault = 0 is normal. */
kve_status kv_evict_plan_set_debug(kve_plan* plan, uint64_t wait_limit_ns,
                                   int32_t fault);

/* Steps 1-2: window attention (Section 3.1 and Eq. 1 context: softmax of the
 * scaled window-query/key logits over the whole causal prefix, window keys
 * included), then per token mu (Eq. 1) and sigma (Eq. 3, divisor n - 1; sigma = 0
 * when n = 1) for every token 0 .. L_r - 1 of every unit. Reads q_win and k,
 * writes mu and sigma, uses ws as scratch. */
kve_status kv_evict_score(const kve_plan* plan, const uint16_t* q_win,
                          const uint16_t* k, float* mu, float* sigma, void* ws,
                          void* stream);

/* Steps 1-2 as kv_evict_score when the softmax normaliser of every window row is
 * already known -- a prefill attention kernel computes it for its own output (Section
 * 3.2 scores with the prefill's existing attention). lse [N_L][n_req][Hq][W] fp32 in
 * q_win's row order (device memory) holds, for the row at position L_r - W + w,
 *   lse = ln sum_{i <= L_r - W + w} exp(q . k_i / sqrt(d))   (natural log),
 * so that A[r][i] = exp(q . k_i / sqrt(d) - lse). The library then needs only the
 * column pass of Eq. 1 and Eq. 3 over the prefix: one pass of the score kernel
 * instead of two. mu and sigma are exactly as accurate as lse is; a row's lse that is
 * not finite makes its terms undefined. Reads q_win, k and lse; writes mu and sigma;
 * uses ws as scratch. */
kve_status kv_evict_score_lse(const kve_plan* plan, const uint16_t* q_win,
                              const uint16_t* k, const float* lse, float* mu,
                              float* sigma, void* ws, void* stream);

/* Steps 1-2 as kv_evict_score, together with the window rows' own attention output.
 * Section 3.2 scores the tokens with the prefill's existing attention; the window rows'
 * attention (the last W positions of every query head) is computed here anyway, so in
 * the same pass over the prefix the library also streams V and returns
 *   O[r] = sum_i A[r][i] * v_i      (A of Eq. 1: causal softmax over the prefix)
 * for every window row, and a caller's prefill can skip attention for those rows.
 * o_win has q_win's layout, [N_L][n_req][Hq][W][d] bf16 (with KVE_PLAN_PER_QUERY_HEAD
 * the same). v follows the plan's v strides. mu and sigma are those of kv_evict_score.
 * Precision: A enters the value product as bf16 (relative error <= 2^-8 per
 * probability), accumulated in fp32, and O is rounded to bf16 once, so
 * |O - O_exact| <= 2^-8 (sum_i A[r][i] |v_i| + |O|) elementwise. attn_ws is a
 * second scratch buffer (256-byte aligned) of kv_evict_score_attn_workspace bytes
 * (fp32 partial outputs, 64 KB per score work item). v must be 128-byte aligned. */
kve_status kv_evict_score_attn(const kve_plan* plan, const uint16_t* q_win,
                               const uint16_t* k, const uint16_t* v, float* mu,
                               float* sigma, uint16_t* o_win, void* ws,
                               void* attn_ws, void* stream);

/* *bytes = the attn_ws size of kv_evict_score_attn for this plan. */
kve_status kv_evict_score_attn_workspace(const kve_plan* plan, size_t* bytes);

/* Step 3: pooling (Section 3.1), base score (Eq. 2), top factor*B candidate pool
 * (Section 3.2), normalisation (Eq. 5, denominator clamped to norm_eps), greedy
 * admission by s~ + lambda2 * corr(i, S) (Eq. 4, Eq. 5) with ties broken towards
 * the lower token position. lambda1 and lambda2 are HOST arrays [N_L] (the
 * layer-wise coefficients of Section 3.3). Writes indices; order and margins may
 * be NULL. Uses ws as scratch. */
kve_status kv_evict_select(const kve_plan* plan, const float* mu,
                           const float* sigma, const uint16_t* k,
                           const float* lambda1, const float* lambda2,
                           int32_t* indices, int32_t* order, float* margins,
                           void* ws, void* stream);

/* Steps 3 and 4 in one launch: exactly what kv_evict_select followed by
 * kv_evict_gather writes (indices, order, margins, k_out, v_out; the same arguments
 * and the same layouts), with the compact cache written by the selection's own CTA
 * for each unit: the kept key rows come from the copy the selection stages for its
 * cosines (Eq. 4), so only the values and the window rows are read again. v may be
 * page-locked host memory as for kv_evict_gather (and k as well). Returns KVE_EINVAL
 * on the conditions of either call. For a plan whose selection runs over every
 * candidate (candidate_factor 0 beyond 512 prefix tokens) the two steps stay two
 * launches. */
kve_status kv_evict_select_gather(const kve_plan* plan, const float* mu,
                                  const float* sigma, const uint16_t* k,
                                  const uint16_t* v, const float* lambda1,
                                  const float* lambda2, int32_t* indices,
                                  int32_t* order, float* margins,
                                  uint16_t* k_out, uint16_t* v_out, void* ws,
                                  void* stream);

/* Step 3 for n_profiles profiles of the layer-wise coefficients in one pass over
 * the units (Section 3.3 searches over profiles and re-selects for each; mu and
 * sigma do not depend on the coefficients, so one kv_evict_score serves them all).
 * lambda1 and lambda2 are HOST arrays [n_profiles][N_L]; profile p selects exactly
 * what kv_evict_select selects with lambda1 + p*N_L and lambda2 + p*N_L. Outputs are
 * stacked by profile: indices [n_profiles][n_units][B]; order and margins likewise
 * (either may be NULL). ws is a separate scratch buffer (256-byte aligned) of
 * kv_evict_select_profiles_workspace bytes, not the plan's workspace; its first word
 * is this call's error word (cleared by the call, read by kv_evict_status(plan, ws,
 * stream)). One launch
 * carries 6144 / (2 N_L) profiles (96 for N_L = 32); more go to further launches on
 * stream. Returns KVE_EINVAL for n_profiles < 1 or a non-finite coefficient, before
 * any launch. */
kve_status kv_evict_select_profiles(const kve_plan* plan, int32_t n_profiles,
                                    const float* mu, const float* sigma,
                                    const uint16_t* k, const float* lambda1,
                                    const float* lambda2, int32_t* indices,
                                    int32_t* order, float* margins, void* ws,
                                    void* stream);

/* *bytes = scratch of kv_evict_select_profiles for n_profiles profiles: a 256-byte
 * header holding the error word, then 4 bytes per prefix token per unit per profile. */
kve_status kv_evict_select_profiles_workspace(const kve_plan* plan,
                                              int32_t n_profiles, size_t* bytes);

/* Step 3 without a workspace. The paper has no counterpart: this entry point
 * exists for callers that cannot allocate device memory at eviction time --
 * serving engines that reserve nearly all of HBM for their own KV-cache pool and
 * hand kernels only pointers into it, or plugin hosts that give a kernel nothing
 * but its inputs and outputs. It computes exactly what kv_evict_select computes,
 * with the same arguments except ws; its scratch (4 bytes per prefix token per
 * unit) is a 16 MiB array compiled into the library, which every GPU that loads
 * the library keeps reserved until the process exits. It allocates nothing.
 *  * Returns KVE_EINVAL when N_L * U * SL exceeds 4194304 (16 MiB / 4 B), where U
 *    is the number of units per layer: Hkv, or Hq for a KVE_PLAN_PER_QUERY_HEAD
 *    plan. E.g. a 32-layer, 8-KV-head request of more than 16384 tokens, or a
 *    per-query-head plan with 32 layers and 32 query heads beyond 4096 tokens.
 *  * Device-side check failures go to an error word that the library keeps beside
 *    the array: kv_evict_status(plan, NULL, stream) reads and clears it.
 *  * The first call on a device looks up the array's device address on that
 *    device (cudaGetSymbolAddress); make that first call before any stream
 *    capture on the device.
 *  * All calls share the one array and each call overwrites it before reading it.
 *    Calls whose executions overlap on the GPU (for example on two streams at
 *    once) race on it and give undefined results; serialise them. */
kve_status kv_evict_select_noalloc(const kve_plan* plan, const float* mu,
                                   const float* sigma, const uint16_t* k,
                                   const float* lambda1, const float* lambda2,
                                   int32_t* indices, int32_t* order,
                                   float* margins, void* stream);

/* Step 4: compact cache (Section 1: each layer keeps B entries after prefill;
 * the window tokens are kept as well). Copies key/value rows bit-exactly.
 * Exception to the device-memory convention: k and v may also be page-locked
 * host memory of the CUDA runtime (cudaHostAlloc, cudaMallocHost, or host memory
 * registered with cudaHostRegister). Under unified addressing the kernel reads
 * such memory in place, and only the kept rows (min(B_l, Lc_r) + W per unit)
 * cross the host link. k_out and v_out stay in device memory. Returns KVE_EINVAL
 * for host memory the runtime does not know (pageable memory) or a pointer the
 * runtime cannot classify. */
kve_status kv_evict_gather(const kve_plan* plan, const uint16_t* k,
                           const uint16_t* v, const int32_t* indices,
                           uint16_t* k_out, uint16_t* v_out, void* stream);

/* Synchronise the stream, read the device error word of ws and clear it. ws is the
 * plan's workspace, the scratch of kv_evict_select_profiles, or NULL for the error
 * word of kv_evict_select_noalloc on the current device.
 * Returns KVE_OK, KVE_ETIMEOUT (a bounded wait ran out) or KVE_ECUDA (a CUDA call
 * failed, or a device-side consistency check of the selection failed: a candidate
 * pool that did not hold exactly C positions -- that unit then reports no
 * selection, indices -1 -- or a pool position outside the unit, whose key row is
 * then not read). */
kve_status kv_evict_status(const kve_plan* plan, void* ws, void* stream);

/* Depth profile of Eq. 6 on the host: kind 0 Global (lambda = sinh(c[0]) on every
 * layer), 1 Segments (sinh(c[0]), sinh(c[1]), sinh(c[2]) on layers
 * [0, b0), [b0, b1), [b1, N_L), with seg_bounds = {b0, b1}, or thirds when
 * seg_bounds is NULL), 2 Curve (sinh(c0 + c1 t + c2 t^2), t = l / (N_L - 1)).
 * Writes lambda_out[num_layers]. */
kve_status kv_evict_profile(int32_t kind, const float* c, int32_t num_layers,
                            const int32_t* seg_bounds, float* lambda_out);

/* A depth-decreasing budget schedule with the total of the uniform one (Section 3.1
 * states only these two properties of PyramidKV's allocation; this function is a
 * reading of it): budgets_out[l] (HOST, [num_layers]) falls linearly with depth
 * from 2B - b to b, b = max(1, floor(last_ratio * B)), rounded down and the
 * remainder given one each to the shallowest layers, so that the budgets are
 * non-increasing and sum to num_layers * B. last_ratio = 1 is uniform. The
 * largest budget is budgets_out[0]: pass it as cfg->budget. Returns KVE_EINVAL
 * unless B >= 1, num_layers >= 1 and 0 < last_ratio <= 1. */
kve_status kv_evict_budget_pyramid(int32_t budget, int32_t num_layers,
                                   float last_ratio, int32_t* budgets_out);

const char* kv_evict_strerror(kve_status status);

#ifdef __cplusplus
}
#endif

#endif /* KV_EVICT_H */
