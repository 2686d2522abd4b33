// Internal declarations of the kv_evict library: the host plan, kernel parameter
// blocks and the unit / work-item geometry shared by host and device code.
#pragma once

#include <cstddef>
#include <cstdint>
#include <utility>
#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/kv_evict.h"

namespace kve {

constexpr int kHeadDim = 128;      // d supported by this build
constexpr int kTileKeys = 128;     // keys per MMA tile (one TMEM accumulator)
constexpr int kSplitTiles = 8;     // most tiles in one work item
constexpr int kMaxRows = 128;      // n = G*W window rows per unit, padded to one M tile
constexpr int kMaxReq = 64;        // requests per call
constexpr int kMaxLayers = 256;    // layers per call (lambda arrays ride in kernel params)
constexpr int kMaxPoolCand = 512;  // candidate pool of the pooled selector (shared memory)
constexpr int kMaxAllCand = 32768; // candidates of the every-candidate selector (Lc)
constexpr int kMaxAllBudget = 1024;// admissions of the every-candidate selector
// Bits of the workspace error word (kv_evict_status).
constexpr uint32_t kErrWait = 1u;    // a bounded wait ran out
constexpr uint32_t kErrCheck = 2u;   // a device-side consistency check failed

// Request table and derived counts, identical on host and device.
struct Geometry {
  int32_t n_req, num_layers, hq, hkv, group, window, n_rows;
  int32_t uheads;                       // heads per layer that own a unit: hkv, or hq
                                        // when every query head selects for itself
  int32_t ugroup;                       // query heads per unit: group, or 1
  int64_t total_tokens;                 // SL
  // element strides of k and v between layers, KV heads and tokens (a row is d
  // contiguous elements); the dense default is token d, head SL*d, layer Hkv*SL*d
  int64_t k_sl, k_sh, k_st;
  int64_t v_sl, v_sh, v_st;
  int64_t n_units;                      // n_req * N_L * uheads
  int64_t n_items;                      // score work items (sum over units of splits)
  int32_t req_len[kMaxReq];             // L_r
  int64_t req_tok_off[kMaxReq];         // off_r
  int32_t req_tiles[kMaxReq];           // ceil(L_r / kTileKeys)
  int32_t req_splits[kMaxReq];          // work items per unit (<= req_tiles)
  int64_t req_unit_base[kMaxReq + 1];   // first unit of request r
  int64_t req_item_base[kMaxReq + 1];   // first item of request r
};

struct UnitInfo {
  int64_t unit;        // (r, l, h) flattened, request-major
  int32_t r, layer, h;
  int32_t L;           // prefix length
  int32_t tiles;       // ceil(L / kTileKeys)
  int32_t splits;      // items of this unit
  int64_t local;       // unit index within its request
  int64_t q_row0;      // first window row in q_win viewed as [rows][d]
  int32_t kvh;         // the KV head whose keys the unit reads
  int64_t tok0;        // token index of the unit's first key in k / v (off_r)
  int64_t k_off;       // element offset of the unit's first key row in k: key i at k_off + i * k_st
  int64_t v_off;       // the same in v
  int64_t mu_off;      // first element of this unit in mu / sigma
  int64_t item0;       // first score item of this unit
};

__host__ __device__ inline UnitInfo unit_info(const Geometry& g, int64_t unit) {
  int r = 0;
  while (r + 1 < g.n_req && g.req_unit_base[r + 1] <= unit) ++r;
  UnitInfo u;
  u.unit = unit;
  u.r = r;
  const int64_t local = unit - g.req_unit_base[r];
  u.layer = static_cast<int32_t>(local / g.uheads);
  u.h = static_cast<int32_t>(local % g.uheads);   // KV head (or query head) of the unit
  u.L = g.req_len[r];
  u.tiles = g.req_tiles[r];
  u.splits = g.req_splits[r];
  u.local = local;
  u.q_row0 = ((static_cast<int64_t>(u.layer) * g.n_req + r) * g.hq +
              static_cast<int64_t>(u.h) * g.ugroup) * g.window;
  const int kvh = g.ugroup == g.group ? u.h : u.h / g.group;   // the KV head the unit reads
  u.kvh = kvh;
  u.tok0 = g.req_tok_off[r];
  u.k_off = u.layer * g.k_sl + kvh * g.k_sh + u.tok0 * g.k_st;
  u.v_off = u.layer * g.v_sl + kvh * g.v_sh + u.tok0 * g.v_st;
  u.mu_off = static_cast<int64_t>(g.num_layers) * g.uheads * g.req_tok_off[r] + local * u.L;
  u.item0 = g.req_item_base[r] + local * u.splits;
  return u;
}

// Score item p (0 <= p < n_items) -> unit and split index.
__host__ __device__ inline int64_t item_unit(const Geometry& g, int64_t p, int32_t* split) {
  int r = 0;
  while (r + 1 < g.n_req && g.req_item_base[r + 1] <= p) ++r;
  const int64_t local = p - g.req_item_base[r];
  *split = static_cast<int32_t>(local % g.req_splits[r]);
  return g.req_unit_base[r] + local / g.req_splits[r];
}

// Tiles [*t0, *t0 + *nt) of item `split` of unit u. The unit's tiles are cut into
// u.splits near-equal runs; the run index is rotated by the unit index so that a
// CTA that always holds the same split index does not always get the longer runs.
__host__ __device__ inline void item_range(const UnitInfo& u, int split, int* t0, int* nt) {
  const int64_t s = (split + u.local) % u.splits;
  const int64_t a = s * u.tiles / u.splits;
  const int64_t b = (s + 1) * u.tiles / u.splits;
  *t0 = static_cast<int>(a);
  *nt = static_cast<int>(b - a);
}

// Workspace layout (byte offsets from the caller's workspace pointer).
struct WsLayout {
  size_t hdr;        // uint32 err
  size_t counts;     // uint32 [n_units]  row-statistics arrivals per unit
  size_t beta;       // uint64 [n_units][kMaxRows]  (log2 softmax normaliser, ready tag)
  size_t clear_end;  // bytes from 0 cleared before each score call
  size_t partial;    // float2 [n_items][kMaxRows]  per-item (max, sum) in log2 units
  size_t keys;       // uint32 [sum of unit lengths]  ordered base scores (select)
  size_t corr;       // float2 [sum of unit lengths]  (corr, 1/|k|): every-candidate selector only
  size_t total;
};

struct ScoreParams {
  Geometry g;
  float alpha;               // log2(e) / sqrt(d)
  uint64_t wait_limit_ns;
  int32_t fault;             // test hook: 1 = unit 0 never publishes its statistics
  int32_t lag;               // rounds a CTA's phase-1 item trails its phase-0 item
  float* mu;
  float* sigma;
  uint32_t* err;
  uint32_t* counts;
  float2* partial;
  unsigned long long* beta;   // low word: beta bits, high word: 1 once written
  float* o_part;              // window output: fp32 [n_items][kMaxRows][d] per column item
  const float* lse;           // given normalisers: natural-log softmax normaliser of every window
                              // row in q_win's row order (the column pass only), or null
};

struct SelectParams {
  Geometry g;
  int32_t budget;            // row stride of indices / order / margins (the plan's B)
  int32_t pool_kernel, cand_factor;
  float norm_eps;
  const float* mu;
  const float* sigma;
  const uint16_t* k;
  int32_t* indices;
  int32_t* order;
  float* margins;
  uint32_t* keys;            // workspace scratch
  uint32_t* err;             // error word read by kv_evict_status: kErrCheck = the pool did not
                             // hold exactly C positions, or a pool position outside the unit
  float* corr;               // workspace scratch of the every-candidate selector (or null):
                             // float2 (corr, 1/|k|) per prefix token of every unit
  const uint16_t* v;         // with k_out and v_out: the selection also writes the compact
  uint16_t* k_out;           // cache of step 4 (as the gather kernel does), or null
  uint16_t* v_out;
  float lambda1[kMaxLayers];
  float lambda2[kMaxLayers];
  int32_t layer_budget[kMaxLayers];   // B_l <= budget kept candidates of layer l
};

// Coefficient profiles of one multi-profile selection launch (kernel parameter):
// profile first + y of the launch (grid y) uses lam[2*y*N_L + l] (lambda1) and
// lam[(2*y + 1)*N_L + l] (lambda2) on layer l, scratch keys + (first + y) *
// keys_stride and outputs + (first + y) * out_stride.
constexpr int kProfileLambdas = 6144;   // 24 KB of coefficients per launch
struct ProfileTable {
  static constexpr bool kMulti = true;
  int32_t first;
  int32_t pad;
  int64_t keys_stride;       // scratch words per profile
  int64_t out_stride;        // output elements per profile (n_units * B)
  float lam[kProfileLambdas];
};

struct GatherParams {
  Geometry g;
  int32_t budget;            // row stride: B + W rows per unit
  int32_t layer_budget[kMaxLayers];
  const uint16_t* k;
  const uint16_t* v;
  const int32_t* indices;
  uint16_t* k_out;
  uint16_t* v_out;
};

}  // namespace kve

struct kve_plan {
  kve_config cfg;
  int32_t layer_budget[kve::kMaxLayers];   // B_l per layer (all cfg.budget by default)
  kve::Geometry geo;
  kve::WsLayout ws;
  uint64_t wait_limit_ns;
  int32_t fault;
  int32_t select_all;   // 1: candidate_factor = 0 and some Lc exceeds kMaxPoolCand, so the
                        // selection runs on the every-candidate selector
};

namespace kve {
// Programmatic dependent launch: a kernel launched with launch_after_previous may be
// scheduled while the previous kernel on its stream finishes; it waits here, before
// touching memory, until that kernel has completed and its writes are visible (a no-op
// for a kernel launched without the attribute).
__device__ __forceinline__ void wait_previous_kernel() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launch `fn` on `stream` after the previous kernel of the stream, overlapping its
// launch with that kernel's tail (programmatic stream serialization).
template <class... KArgs, class... Args>
cudaError_t launch_after_previous(void (*fn)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                  cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fn, std::forward<Args>(args)...);
}

// Kernel launchers (defined next to their kernels).
// tm_v = null: the plain score kernel; otherwise the variant that also accumulates the
// window rows' attention output into p.o_part (then launch_attn_finish).
cudaError_t launch_score(const kve_plan& plan, const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                         const CUtensorMap* tm_v, const ScoreParams& p, int ctas, cudaStream_t stream);
cudaError_t launch_attn_finish(const kve_plan& plan, const float* o_part, uint16_t* o_win,
                               cudaStream_t stream);
cudaError_t launch_select(const kve_plan& plan, const SelectParams& p, cudaStream_t stream);
cudaError_t launch_select_all(const kve_plan& plan, const SelectParams& p, cudaStream_t stream);
cudaError_t launch_select_profiles(const kve_plan& plan, const SelectParams& p, const ProfileTable& table,
                                   int profiles, cudaStream_t stream);
cudaError_t launch_gather(const kve_plan& plan, const GatherParams& p, cudaStream_t stream);

// The select kernel's parameters common to every selection entry point (host code,
// kve_host.cu); lambda1 / lambda2 (HOST [N_L]) may be NULL when a profile table
// supplies the coefficients. Leaves keys, err and corr null.
kve_status select_params(const kve_plan* plan, const float* mu, const float* sigma, const uint16_t* k,
                         const float* lambda1, const float* lambda2, int32_t* indices, int32_t* order,
                         float* margins, SelectParams* p);

// Device address, on the current device, of the error word of the selection that
// runs without a workspace (kve_select.cu); null when it cannot be looked up.
uint32_t* noalloc_error_word();
}  // namespace kve
