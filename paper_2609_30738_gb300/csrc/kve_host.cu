// Host side of the kv_evict C ABI: plan validation and work geometry, workspace
// layout, TMA descriptor encoding and the launches of the three kernels.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>

#include <cudaTypedefs.h>

#include "kve_internal.h"

namespace {

using kve::kHeadDim;
using kve::kMaxLayers;
using kve::kMaxReq;
using kve::kMaxRows;
using kve::kSplitTiles;
using kve::kTileKeys;

constexpr uint64_t kDefaultWaitNs = 2000000000ull;   // 2 s

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// [rows][128] bf16 viewed as a 2-D tensor; boxes of 64 elements x 128 rows with the
// 128-byte swizzle, rows past the end read as zero.
bool encode_rows(CUtensorMap* map, const void* base, int64_t rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(kHeadDim) * 2};
  cuuint32_t box[2] = {64, 128};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// k (or v) viewed as a 4-D tensor (d, token, KV head, layer) with the plan's element
// strides; boxes of 64 elements x 128 tokens with the 128-byte swizzle, tokens past SL
// read as zero.
bool encode_keys(CUtensorMap* map, const void* base, const kve::Geometry& g, bool values = false) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(g.total_tokens),
                        static_cast<cuuint64_t>(g.hkv), static_cast<cuuint64_t>(g.num_layers)};
  const int64_t st = values ? g.v_st : g.k_st, sh = values ? g.v_sh : g.k_sh, sl = values ? g.v_sl : g.k_sl;
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(st) * 2, static_cast<cuuint64_t>(sh) * 2,
                           static_cast<cuuint64_t>(sl) * 2};
  cuuint32_t box[4] = {64, 128, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int device_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

// Score items per unit for a unit of T tiles. Items hold at most kSplitTiles tiles.
// The score kernel deals items to its CTAs round-robin, one round = one item per CTA,
// so a split count that divides the CTA count (or is a multiple of it) makes every
// round hold whole units; up to twice the minimum count is accepted for that.
int32_t choose_splits(int64_t T, int64_t ctas) {
  const int64_t kmin = (T + kSplitTiles - 1) / kSplitTiles;
  const int64_t kmax = std::min<int64_t>(T, 2 * kmin);
  for (int64_t k = kmin; ctas > 0 && k <= kmax; ++k)
    if (ctas % k == 0 || k % ctas == 0) return static_cast<int32_t>(k);
  return static_cast<int32_t>(kmin);
}

// Rounds a CTA's phase-1 item trails its phase-0 item in the score kernel: one more
// than the most rounds any unit's items span. Any lag at least that span is free of
// circular waits; the extra round gives a unit's merge time to land before its first
// phase-1 item, while the K tiles streamed in between (two rounds, about 64 MB at full
// width) stay in L2 for the phase-1 re-read.
int32_t score_lag(const kve::Geometry& g, int64_t ctas) {
  int64_t span = 0;
  const int64_t units_per_req = static_cast<int64_t>(g.num_layers) * g.uheads;
  for (int r = 0; r < g.n_req; ++r) {
    const int64_t k = g.req_splits[r];
    // (first item) mod ctas repeats with period ctas / gcd(k, ctas) <= ctas
    const int64_t n = std::min<int64_t>(units_per_req, ctas);
    for (int64_t ul = 0; ul < n; ++ul) {
      const int64_t a = g.req_item_base[r] + ul * k;
      span = std::max<int64_t>(span, (a + k - 1) / ctas - a / ctas);
    }
  }
  return static_cast<int32_t>(span + 1);
}

}  // namespace

extern "C" {

kve_status kv_evict_plan(const kve_config* cfg, const int64_t* seq_lens, int32_t n_req,
                         kve_plan** plan_out, size_t* workspace_bytes) {
  return kv_evict_plan_layered(cfg, seq_lens, n_req, nullptr, plan_out, workspace_bytes);
}

kve_status kv_evict_plan_layered(const kve_config* cfg, const int64_t* seq_lens, int32_t n_req,
                                 const int32_t* layer_budgets, kve_plan** plan_out,
                                 size_t* workspace_bytes) {
  return kv_evict_plan_ex(cfg, seq_lens, n_req, layer_budgets, 0, plan_out, workspace_bytes);
}

kve_status kv_evict_plan_ex(const kve_config* cfg, const int64_t* seq_lens, int32_t n_req,
                            const int32_t* layer_budgets, int32_t flags, kve_plan** plan_out,
                            size_t* workspace_bytes) {
  if (!cfg || !seq_lens || !plan_out) return KVE_EINVAL;
  if ((flags & ~KVE_PLAN_PER_QUERY_HEAD) != 0) return KVE_EINVAL;
  *plan_out = nullptr;
  const kve_config& c = *cfg;
  if (c.num_layers < 1 || c.num_layers > kMaxLayers) return KVE_EINVAL;
  if (c.num_kv_heads < 1 || c.num_q_heads < c.num_kv_heads || c.num_q_heads % c.num_kv_heads) return KVE_EINVAL;
  if (c.head_dim != kHeadDim) return KVE_EINVAL;
  const int G = c.num_q_heads / c.num_kv_heads;
  if (c.window < 1 || static_cast<int64_t>(G) * c.window > kMaxRows) return KVE_EINVAL;
  if (c.budget < 1 || c.pool_kernel < 1 || c.pool_kernel > 255 || c.pool_kernel % 2 == 0)
    return KVE_EINVAL;
  if (c.candidate_factor < 0 || !(c.norm_eps > 0.f) || !std::isfinite(c.norm_eps)) return KVE_EINVAL;
  if (n_req < 1 || n_req > kMaxReq) return KVE_EINVAL;

  kve_plan* plan = new (std::nothrow) kve_plan;
  if (!plan) return KVE_ENOMEM;
  std::memset(plan, 0, sizeof(*plan));
  plan->cfg = c;
  for (int l = 0; l < c.num_layers; ++l) {
    const int32_t b = layer_budgets ? layer_budgets[l] : c.budget;
    if (b < 1 || b > c.budget) {
      delete plan;
      return KVE_EINVAL;
    }
    plan->layer_budget[l] = b;
  }
  plan->wait_limit_ns = kDefaultWaitNs;
  plan->fault = 0;
  kve::Geometry& g = plan->geo;
  g.n_req = n_req;
  g.num_layers = c.num_layers;
  g.hq = c.num_q_heads;
  g.hkv = c.num_kv_heads;
  g.group = G;
  g.window = c.window;
  const bool per_q = (flags & KVE_PLAN_PER_QUERY_HEAD) != 0;
  g.uheads = per_q ? c.num_q_heads : c.num_kv_heads;
  g.ugroup = per_q ? 1 : G;
  g.n_rows = g.ugroup * c.window;
  int64_t off = 0, units = 0, items = 0, max_lc = 0;
  const int64_t units_per_req = static_cast<int64_t>(c.num_layers) * g.uheads;
  int ctas = device_sms();
  if (ctas <= 0) {
    cudaGetLastError();
    ctas = 152;   // no device visible: plan for a full GB300
  }
  for (int r = 0; r < n_req; ++r) {
    const int64_t L = seq_lens[r];
    if (L <= c.window || L > (int64_t(1) << 30)) {
      delete plan;
      return KVE_EINVAL;
    }
    g.req_len[r] = static_cast<int32_t>(L);
    g.req_tok_off[r] = off;
    g.req_tiles[r] = static_cast<int32_t>((L + kTileKeys - 1) / kTileKeys);
    g.req_splits[r] = choose_splits(g.req_tiles[r], ctas);
    g.req_unit_base[r] = units;
    g.req_item_base[r] = items;
    off += L;
    units += units_per_req;
    items += units_per_req * g.req_splits[r];
    if (L - c.window > max_lc) max_lc = L - c.window;
  }
  g.req_unit_base[n_req] = units;
  g.req_item_base[n_req] = items;
  g.total_tokens = off;
  // the dense layouts [N_L][Hkv][SL][d] until kv_evict_plan_set_kv_strides
  g.k_st = g.v_st = kHeadDim;
  g.k_sh = g.v_sh = off * kHeadDim;
  g.k_sl = g.v_sl = static_cast<int64_t>(c.num_kv_heads) * off * kHeadDim;
  g.n_units = units;
  g.n_items = items;
  const int64_t max_cand = c.candidate_factor == 0 ? max_lc
                                                   : std::min<int64_t>(int64_t(c.candidate_factor) * c.budget, max_lc);
  // TMA coordinates (window rows of q_win, tokens of k) are 32-bit; the select kernel
  // holds its pool in shared memory
  const int64_t q_rows = static_cast<int64_t>(c.num_layers) * n_req * c.num_q_heads * c.window;
  // candidate_factor = 0 beyond the pooled selector's pool runs the every-candidate
  // selector (Lc <= kMaxAllCand, B <= kMaxAllBudget)
  plan->select_all = (c.candidate_factor == 0 && max_lc > kve::kMaxPoolCand) ? 1 : 0;
  const bool cand_ok = plan->select_all ? (max_lc <= kve::kMaxAllCand && c.budget <= kve::kMaxAllBudget)
                                        : max_cand <= kve::kMaxPoolCand;
  if (!cand_ok || off >= (int64_t(1) << 31) - 256 || q_rows >= (int64_t(1) << 31) - 256 ||
      2 * items >= (int64_t(1) << 31) || units >= (int64_t(1) << 31)) {
    delete plan;
    return KVE_EINVAL;
  }
  kve::WsLayout& w = plan->ws;
  w.hdr = 0;
  w.counts = 256;
  w.beta = align_up(w.counts + 4 * units, 256);
  w.clear_end = align_up(w.beta + sizeof(uint64_t) * kMaxRows * units, 256);
  w.partial = w.clear_end;
  w.keys = align_up(w.partial + sizeof(float2) * kMaxRows * items, 256);
  w.corr = plan->select_all ? align_up(w.keys + sizeof(uint32_t) * units_per_req * off, 256) : 0;
  w.total = plan->select_all ? align_up(w.corr + sizeof(float2) * units_per_req * off, 256)
                              : align_up(w.keys + sizeof(uint32_t) * units_per_req * off, 256);
  if (workspace_bytes) *workspace_bytes = w.total;
  *plan_out = plan;
  return KVE_OK;
}

void kv_evict_plan_destroy(kve_plan* plan) { delete plan; }

kve_status kv_evict_plan_set_kv_strides(kve_plan* plan, const int64_t* k_strides, const int64_t* v_strides) {
  if (!plan) return KVE_EINVAL;
  kve::Geometry& g = plan->geo;
  const int64_t dense[3] = {static_cast<int64_t>(g.hkv) * g.total_tokens * kHeadDim, g.total_tokens * kHeadDim,
                            kHeadDim};
  const int64_t* ks = k_strides ? k_strides : dense;
  const int64_t* vs = v_strides ? v_strides : dense;
  // each stride a multiple of 8 elements (16 bytes, the TMA and vector-load rule) and
  // below 2^37 elements (TMA strides below 2^40 bytes); a token step of at least one row
  for (const int64_t* st : {ks, vs}) {
    for (int i = 0; i < 3; ++i)
      if (st[i] < 0 || st[i] % 8 != 0 || st[i] >= (int64_t(1) << 37)) return KVE_EINVAL;
    if (st[2] < kHeadDim) return KVE_EINVAL;
  }
  g.k_sl = ks[0];
  g.k_sh = ks[1];
  g.k_st = ks[2];
  g.v_sl = vs[0];
  g.v_sh = vs[1];
  g.v_st = vs[2];
  return KVE_OK;
}

kve_status kv_evict_plan_set_debug(kve_plan* plan, uint64_t wait_limit_ns, int32_t fault) {
  if (!plan || wait_limit_ns == 0 || fault < 0 || fault > 1) return KVE_EINVAL;
  plan->wait_limit_ns = wait_limit_ns;
  plan->fault = fault;
  return KVE_OK;
}

}  // extern "C"

namespace {

// The score step, with the window output when v is given (o_win, attn_ws then too).
kve_status score_impl(const kve_plan* plan, const uint16_t* q_win, const uint16_t* k, const uint16_t* v,
                      float* mu, float* sigma, uint16_t* o_win, void* ws, void* attn_ws, void* stream,
                      const float* lse = nullptr) {
  if (!plan || !q_win || !k || !mu || !sigma || !ws) return KVE_EINVAL;
  if (lse && (v || !aligned(lse, 4))) return KVE_EINVAL;
  if (!aligned(q_win, 128) || !aligned(k, 128) || !aligned(mu, 16) || !aligned(sigma, 16) || !aligned(ws, 256))
    return KVE_EINVAL;
  if (v && (!o_win || !attn_ws || !aligned(v, 128) || !aligned(o_win, 16) || !aligned(attn_ws, 256)))
    return KVE_EINVAL;
  const kve::Geometry& g = plan->geo;
  const int sms = device_sms();
  if (sms <= 0) return KVE_ECUDA;
  CUtensorMap tm_q, tm_k, tm_v;
  const int64_t q_rows = static_cast<int64_t>(g.num_layers) * g.n_req * g.hq * g.window;
  if (!encode_rows(&tm_q, q_win, q_rows) || !encode_keys(&tm_k, k, g)) return KVE_ECUDA;
  if (v && !encode_keys(&tm_v, v, g, true)) return KVE_ECUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* w = static_cast<uint8_t*>(ws);
  if (cudaMemsetAsync(w, 0, plan->ws.clear_end, st) != cudaSuccess) return KVE_ECUDA;
  kve::ScoreParams p;
  std::memset(&p, 0, sizeof(p));
  p.g = g;
  p.alpha = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(kHeadDim)));
  p.wait_limit_ns = plan->wait_limit_ns;
  p.fault = plan->fault;
  p.mu = mu;
  p.sigma = sigma;
  p.err = reinterpret_cast<uint32_t*>(w);
  p.counts = reinterpret_cast<uint32_t*>(w + plan->ws.counts);
  p.partial = reinterpret_cast<float2*>(w + plan->ws.partial);
  p.beta = reinterpret_cast<unsigned long long*>(w + plan->ws.beta);
  p.o_part = static_cast<float*>(attn_ws);
  p.lse = lse;
  const int64_t ctas = std::min<int64_t>(sms, g.n_items);
  p.lag = score_lag(g, ctas);
  if (kve::launch_score(*plan, tm_q, tm_k, v ? &tm_v : nullptr, p, static_cast<int>(ctas), st) != cudaSuccess)
    return KVE_ECUDA;
  if (v && kve::launch_attn_finish(*plan, p.o_part, o_win, st) != cudaSuccess) return KVE_ECUDA;
  return KVE_OK;
}

}  // namespace

extern "C" {

kve_status kv_evict_score(const kve_plan* plan, const uint16_t* q_win, const uint16_t* k, float* mu,
                          float* sigma, void* ws, void* stream) {
  return score_impl(plan, q_win, k, nullptr, mu, sigma, nullptr, ws, nullptr, stream);
}

kve_status kv_evict_score_lse(const kve_plan* plan, const uint16_t* q_win, const uint16_t* k, const float* lse,
                              float* mu, float* sigma, void* ws, void* stream) {
  if (!lse) return KVE_EINVAL;
  return score_impl(plan, q_win, k, nullptr, mu, sigma, nullptr, ws, nullptr, stream, lse);
}

kve_status kv_evict_score_attn(const kve_plan* plan, const uint16_t* q_win, const uint16_t* k,
                               const uint16_t* v, float* mu, float* sigma, uint16_t* o_win, void* ws,
                               void* attn_ws, void* stream) {
  if (!v) return KVE_EINVAL;
  return score_impl(plan, q_win, k, v, mu, sigma, o_win, ws, attn_ws, stream);
}

kve_status kv_evict_score_attn_workspace(const kve_plan* plan, size_t* bytes) {
  if (!plan || !bytes) return KVE_EINVAL;
  *bytes = align_up(static_cast<size_t>(plan->geo.n_items) * kMaxRows * kHeadDim * sizeof(float), 256);
  return KVE_OK;
}

}  // extern "C"

namespace kve {

kve_status select_params(const kve_plan* plan, const float* mu, const float* sigma, const uint16_t* k,
                         const float* lambda1, const float* lambda2, int32_t* indices, int32_t* order,
                         float* margins, SelectParams* p) {
  const kve::Geometry& g = plan->geo;
  std::memset(p, 0, sizeof(*p));
  p->g = g;
  p->budget = plan->cfg.budget;
  p->pool_kernel = plan->cfg.pool_kernel;
  p->cand_factor = plan->cfg.candidate_factor;
  p->norm_eps = plan->cfg.norm_eps;
  for (int l = 0; l < g.num_layers; ++l) {
    if (lambda1 && (!std::isfinite(lambda1[l]) || !std::isfinite(lambda2[l]))) return KVE_EINVAL;
    p->lambda1[l] = lambda1 ? lambda1[l] : 0.f;
    p->lambda2[l] = lambda2 ? lambda2[l] : 0.f;
    p->layer_budget[l] = plan->layer_budget[l];
  }
  p->mu = mu;
  p->sigma = sigma;
  p->k = k;
  p->indices = indices;
  p->order = order;
  p->margins = margins;
  return KVE_OK;
}

}  // namespace kve

namespace {

using kve::select_params;

// Bytes in front of the multi-profile scratch that hold its error word.
constexpr size_t kProfileHeader = 256;

// Scratch words of one profile (the ordered base score of every prefix token of
// every unit), padded to 256 bytes.
int64_t profile_keys_words(const kve_plan* plan) {
  const kve::Geometry& g = plan->geo;
  const int64_t words = static_cast<int64_t>(g.num_layers) * g.uheads * g.total_tokens;
  return (words + 63) / 64 * 64;
}

// Profiles one launch can carry in its parameter table.
int32_t profiles_per_launch(const kve_plan* plan) {
  return kve::kProfileLambdas / (2 * plan->geo.num_layers);
}

// Sources of the compact cache may be pinned host memory (read in place under unified
// addressing); host memory the CUDA runtime does not know is refused.
bool readable_source(const void* src) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, src) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type != cudaMemoryTypeUnregistered;
}

}  // namespace

extern "C" {

kve_status kv_evict_select(const kve_plan* plan, const float* mu, const float* sigma, const uint16_t* k,
                           const float* lambda1, const float* lambda2, int32_t* indices, int32_t* order,
                           float* margins, void* ws, void* stream) {
  if (!plan || !mu || !sigma || !k || !lambda1 || !lambda2 || !indices || !ws) return KVE_EINVAL;
  if (!aligned(k, 16) || !aligned(mu, 16) || !aligned(sigma, 16) || !aligned(ws, 256)) return KVE_EINVAL;
  kve::SelectParams p;
  const kve_status s = select_params(plan, mu, sigma, k, lambda1, lambda2, indices, order, margins, &p);
  if (s != KVE_OK) return s;
  p.keys = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + plan->ws.keys);
  p.err = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + plan->ws.hdr);
  if (plan->select_all) {
    p.corr = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + plan->ws.corr);
    return kve::launch_select_all(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK
                                                                                              : KVE_ECUDA;
  }
  return kve::launch_select(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK : KVE_ECUDA;
}

kve_status kv_evict_select_gather(const kve_plan* plan, const float* mu, const float* sigma, const uint16_t* k,
                                  const uint16_t* v, const float* lambda1, const float* lambda2,
                                  int32_t* indices, int32_t* order, float* margins, uint16_t* k_out,
                                  uint16_t* v_out, void* ws, void* stream) {
  if (!plan || !mu || !sigma || !k || !v || !lambda1 || !lambda2 || !indices || !k_out || !v_out || !ws)
    return KVE_EINVAL;
  if (!aligned(k, 16) || !aligned(v, 16) || !aligned(k_out, 16) || !aligned(v_out, 16) || !aligned(mu, 16) ||
      !aligned(sigma, 16) || !aligned(ws, 256))
    return KVE_EINVAL;
  if (!readable_source(k) || !readable_source(v)) return KVE_EINVAL;
  if (plan->select_all) {
    // the every-candidate selector keeps its own launch; the gather follows it
    const kve_status s = kv_evict_select(plan, mu, sigma, k, lambda1, lambda2, indices, order, margins, ws,
                                         stream);
    return s != KVE_OK ? s : kv_evict_gather(plan, k, v, indices, k_out, v_out, stream);
  }
  kve::SelectParams p;
  const kve_status s = select_params(plan, mu, sigma, k, lambda1, lambda2, indices, order, margins, &p);
  if (s != KVE_OK) return s;
  p.keys = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + plan->ws.keys);
  p.err = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + plan->ws.hdr);
  p.v = v;
  p.k_out = k_out;
  p.v_out = v_out;
  return kve::launch_select(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK : KVE_ECUDA;
}

kve_status kv_evict_select_profiles_workspace(const kve_plan* plan, int32_t n_profiles, size_t* bytes) {
  if (!plan || !bytes || n_profiles < 1 || plan->select_all) return KVE_EINVAL;
  *bytes = kProfileHeader +
           static_cast<size_t>(n_profiles) * static_cast<size_t>(profile_keys_words(plan)) * sizeof(uint32_t);
  return KVE_OK;
}

kve_status kv_evict_select_profiles(const kve_plan* plan, int32_t n_profiles, const float* mu,
                                    const float* sigma, const uint16_t* k, const float* lambda1,
                                    const float* lambda2, int32_t* indices, int32_t* order, float* margins,
                                    void* ws, void* stream) {
  if (!plan || n_profiles < 1 || !mu || !sigma || !k || !lambda1 || !lambda2 || !indices || !ws ||
      plan->select_all)
    return KVE_EINVAL;
  if (!aligned(k, 16) || !aligned(mu, 16) || !aligned(sigma, 16) || !aligned(ws, 256)) return KVE_EINVAL;
  const int32_t nl = plan->geo.num_layers;
  for (int64_t i = 0; i < static_cast<int64_t>(n_profiles) * nl; ++i)
    if (!std::isfinite(lambda1[i]) || !std::isfinite(lambda2[i])) return KVE_EINVAL;
  kve::SelectParams p;
  const kve_status s = select_params(plan, mu, sigma, k, nullptr, nullptr, indices, order, margins, &p);
  if (s != KVE_OK) return s;
  // the error word (cleared here, read by kv_evict_status on this ws), then the
  // profiles' base-score keys
  if (cudaMemsetAsync(ws, 0, sizeof(uint32_t), static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return KVE_ECUDA;
  p.err = static_cast<uint32_t*>(ws);
  p.keys = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + kProfileHeader);
  // the table rides in the kernel parameters; profiles beyond its capacity go to
  // further launches on the same stream
  static thread_local kve::ProfileTable table;
  table.pad = 0;
  table.keys_stride = profile_keys_words(plan);
  table.out_stride = plan->geo.n_units * static_cast<int64_t>(plan->cfg.budget);
  const int32_t cap = profiles_per_launch(plan);
  for (int32_t f = 0; f < n_profiles; f += cap) {
    const int32_t cnt = std::min(cap, n_profiles - f);
    table.first = f;
    for (int32_t j = 0; j < cnt; ++j)
      for (int32_t l = 0; l < nl; ++l) {
        table.lam[(2 * j) * nl + l] = lambda1[static_cast<int64_t>(f + j) * nl + l];
        table.lam[(2 * j + 1) * nl + l] = lambda2[static_cast<int64_t>(f + j) * nl + l];
      }
    if (kve::launch_select_profiles(*plan, p, table, cnt, static_cast<cudaStream_t>(stream)) != cudaSuccess)
      return KVE_ECUDA;
  }
  return KVE_OK;
}

kve_status kv_evict_gather(const kve_plan* plan, const uint16_t* k, const uint16_t* v, const int32_t* indices,
                           uint16_t* k_out, uint16_t* v_out, void* stream) {
  if (!plan || !k || !v || !indices || !k_out || !v_out) return KVE_EINVAL;
  if (!aligned(k, 16) || !aligned(v, 16) || !aligned(k_out, 16) || !aligned(v_out, 16)) return KVE_EINVAL;
  if (!readable_source(k) || !readable_source(v)) return KVE_EINVAL;
  kve::GatherParams p;
  std::memset(&p, 0, sizeof(p));
  p.g = plan->geo;
  p.budget = plan->cfg.budget;
  for (int l = 0; l < plan->geo.num_layers; ++l) p.layer_budget[l] = plan->layer_budget[l];
  p.k = k;
  p.v = v;
  p.indices = indices;
  p.k_out = k_out;
  p.v_out = v_out;
  return kve::launch_gather(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK : KVE_ECUDA;
}

kve_status kv_evict_status(const kve_plan* plan, void* ws, void* stream) {
  if (!plan) return KVE_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return KVE_ECUDA;
  if (!ws) {
    // the error word of the selection without a workspace, on the current device
    ws = kve::noalloc_error_word();
    if (!ws) return KVE_ECUDA;
  }
  uint32_t err = 0;
  if (cudaMemcpy(&err, ws, sizeof(err), cudaMemcpyDeviceToHost) != cudaSuccess) return KVE_ECUDA;
  if (err != 0) {
    if (cudaMemset(ws, 0, sizeof(err)) != cudaSuccess) return KVE_ECUDA;
    return (err & kve::kErrCheck) ? KVE_ECUDA : KVE_ETIMEOUT;
  }
  return KVE_OK;
}

kve_status kv_evict_profile(int32_t kind, const float* c, int32_t num_layers, const int32_t* seg_bounds,
                            float* lambda_out) {
  if (!c || !lambda_out || num_layers < 1 || kind < 0 || kind > 2) return KVE_EINVAL;
  int b0 = (num_layers + 2) / 3, b1 = (2 * num_layers + 2) / 3;   // ceil(N/3), ceil(2N/3)
  if (seg_bounds) {
    b0 = seg_bounds[0];
    b1 = seg_bounds[1];
    if (b0 < 0 || b1 < b0 || b1 > num_layers) return KVE_EINVAL;
  }
  for (int l = 0; l < num_layers; ++l) {
    double a;
    if (kind == 0) {
      a = c[0];
    } else if (kind == 1) {
      a = l < b0 ? c[0] : (l < b1 ? c[1] : c[2]);
    } else {
      const double t = num_layers > 1 ? static_cast<double>(l) / (num_layers - 1) : 0.0;
      a = static_cast<double>(c[0]) + static_cast<double>(c[1]) * t + static_cast<double>(c[2]) * t * t;
    }
    lambda_out[l] = static_cast<float>(std::sinh(a));
  }
  return KVE_OK;
}

kve_status kv_evict_budget_pyramid(int32_t budget, int32_t num_layers, float last_ratio,
                                   int32_t* budgets_out) {
  if (!budgets_out || budget < 1 || num_layers < 1 || !(last_ratio > 0.f) || last_ratio > 1.f)
    return KVE_EINVAL;
  const int64_t N = num_layers, total = N * budget;
  if (N == 1) {
    budgets_out[0] = budget;
    return KVE_OK;
  }
  // linear in depth from top to bottom = max(1, floor(r*B)), top = 2B - bottom, so the
  // mean is B; the floors' shortfall goes to the shallowest layers, one each
  const int64_t bottom = std::max<int64_t>(1, static_cast<int64_t>(std::floor(last_ratio * budget)));
  const int64_t top = 2 * static_cast<int64_t>(budget) - bottom;
  int64_t sum = 0;
  for (int64_t l = 0; l < N; ++l) {
    // floor of the linear interpolation: never above it, so sum <= total
    const int64_t b = bottom + ((top - bottom) * (N - 1 - l)) / (N - 1);
    budgets_out[l] = static_cast<int32_t>(b);
    sum += b;
  }
  for (int64_t l = 0; sum < total; l = (l + 1) % N, ++sum) ++budgets_out[l];
  return KVE_OK;
}

const char* kv_evict_strerror(kve_status s) {
  switch (s) {
    case KVE_OK: return "ok";
    case KVE_EINVAL: return "invalid argument or unsupported shape";
    case KVE_ECUDA: return "CUDA call failed";
    case KVE_ETIMEOUT: return "device-side wait timed out";
    case KVE_ENOMEM: return "host allocation failed";
  }
  return "unknown status";
}

}  // extern "C"
