// Window-score kernel: steps 1-2 of the eviction step (Section 3.1, Eq. 1, Eq. 3).
//
// For every unit (request, layer, KV head) the n = G*W window rows attend to the
// L prefix keys through a causal softmax; mu_i and sigma_i are the mean and the
// sample standard deviation of A[., i] over the n rows.
//
// Work is cut into items of up to kSplitKeys keys (tiles of 128). Each item runs in
// one of two phases on a persistent, warp-specialised CTA:
//   phase 0 (row statistics):   D[row][key] = Q K^T on tcgen05 (rows on TMEM lanes);
//                               each epilogue thread owns one row and keeps the
//                               running max m and sum Z = sum 2^(alpha*l - m) of its
//                               row; the item's (m, Z) per row are published, and
//                               the last item of a unit to publish merges them into
//                               beta_r = log2 of the row's softmax normaliser and
//                               raises the unit's ready flag.
//   phase 1 (column statistics): D[key][row] = K Q^T (keys on TMEM lanes); each
//                               epilogue thread owns one key, forms
//                               A = 2^(alpha*l - beta_r) for its n rows and reduces
//                               them to mu and sigma in registers (two passes).
// Work is claimed from two queues, both in unit order. A CTA's producer holds one
// claimed phase-1 item and pushes it into the CTA's pipeline only once its unit's
// statistics are merged (a relaxed poll of the unit's done flag, overlapped with
// the loads of the current item); until then it claims phase-0 items. Nothing
// waits on another CTA while phase-0 work remains, so the schedule needs neither an
// ordering argument nor co-residency, and a phase-1 item re-reads its K tiles about
// one merge latency after they were streamed, while they are still in L2. The
// final waits (no phase-0 work left) are bounded and a timeout is reported as
// KVE_ETIMEOUT.
//
// Roles: warp 0 claims items and issues TMA loads; warp 1 owns TMEM and issues the
// MMAs; warp 2 (sync) does all cross-CTA work in claim order -- it publishes the
// row statistics of phase-0 items, merges a unit's statistics when its last item
// arrives, and stages -beta of phase-1 items in shared memory ahead of use; warps
// 3-10 run the epilogue in two groups of four (warp w reads TMEM lanes
// 32*(w%4)..+31), the groups taking alternate tiles. The epilogue warps never
// touch global synchronisation; they only compute, write shared memory and
// arrive on mbarriers.
#include <cstddef>

#include "kve_internal.h"
#include "kve_ptx.cuh"

namespace kve {
namespace {

constexpr int kThreads = 352;
constexpr int kSyncWarp = 2;
constexpr int kEpiWarp0 = 3;
constexpr int kEpiWarps = 8;
constexpr int kQBufs = 2;
constexpr int kKStages = 4;
constexpr int kAccBufs = 4;      // 4 x 128 TMEM columns
constexpr int kItemSlots = 4;
constexpr uint32_t kTileBytes = 128 * kHeadDim * 2;   // 32 KB: 128 rows x 128 bf16
constexpr uint32_t kHalfBytes = kTileBytes / 2;       // one 64-element (128 B) column block
constexpr uint32_t kTmemCols = 512;
constexpr size_t kDynSmem = (kQBufs + kKStages) * kTileBytes + 1024;
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);

struct ScoreCtl {
  uint64_t q_full[kQBufs], q_empty[kQBufs];
  uint64_t k_full[kKStages], k_empty[kKStages];
  uint64_t acc_full[kAccBufs], acc_empty[kAccBufs];
  uint64_t item_full[kItemSlots], item_empty[kItemSlots];
  uint64_t pub_full[kItemSlots];    // epilogue -> sync warp, once per item
  uint64_t beta_full[kItemSlots];   // sync warp -> epilogue, once per item
  int64_t item_ring[kItemSlots];
  uint32_t tmem_base;
  volatile int abort;
  int32_t roww[kMaxRows];                            // r % W
  alignas(16) float2 comb[kItemSlots][2][kMaxRows];  // per group (m, Z) of a row item
  alignas(16) float nbeta[kItemSlots][kMaxRows];     // -beta of a column item
};
static_assert(offsetof(ScoreCtl, nbeta) % 16 == 0, "nbeta is read with 16-byte loads");
static_assert(offsetof(ScoreCtl, comb) % 16 == 0, "comb holds float2");

struct Claim {
  int phase;
  int64_t p;
};

// Ring entry: item index in the low bits, phase in bit 62; -1 ends the work.
__device__ __forceinline__ int64_t encode_claim(int phase, int64_t p) {
  return p | (static_cast<int64_t>(phase) << 62);
}

__device__ __forceinline__ Claim decode_claim(int64_t c) {
  Claim k;
  k.phase = static_cast<int>((c >> 62) & 1);
  k.p = c & ((int64_t(1) << 62) - 1);
  return k;
}

__device__ __forceinline__ int item_tiles(int L, int split) {
  const int left = L - split * kSplitKeys;
  const int t = (left + kTileKeys - 1) / kTileKeys;
  return t < kSplitTiles ? t : kSplitTiles;
}

__device__ __forceinline__ void set_error(const ScoreParams& P, ScoreCtl& ctl, uint32_t code) {
  atomicOr(P.err, code);
  ctl.abort = 1;
}

// Bounded wait whose outcome is the same for every lane of the warp, so that a
// warp never splits in front of a .sync.aligned instruction.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit,
                                          volatile int* abort) {
  const bool ok = mbar_wait(bar, parity, global_timer_ns() + limit, abort);
  return __all_sync(0xffffffffu, ok);
}

// Merge of two (m, Z) pairs in log2 units: Z counts 2^(x - m).
__device__ __forceinline__ float2 merge_mz(float2 a, float2 b) {
  const float m = fmaxf(a.x, b.x);
  if (m == -INFINITY) return make_float2(-INFINITY, 0.f);
  float z = 0.f;
  if (a.x != -INFINITY) z = fmaf(a.y, ex2(a.x - m), z);
  if (b.x != -INFINITY) z = fmaf(b.y, ex2(b.x - m), z);
  return make_float2(m, z);
}

// ---------------------------------------------------------------- epilogue, phase 0

template <bool kFull>
__device__ __forceinline__ bool rowstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, int split, uint32_t slot,
                                              uint32_t& ai) {
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int grp = (threadIdx.x - kEpiWarp0 * 32) >> 7;   // 0 or 1
  const int row = quad * 32 + lane;
  const int W = P.g.window;
  const int lim_all = u.L - W;                 // keys <= lim_all are seen by every row
  const int lim = u.L - W + ctl.roww[row];     // last key this row sees
  const int ntiles = item_tiles(u.L, split);
  const float alpha = P.alpha;
  float m = -INFINITY, Z = 0.f;
  for (int t = 0; t < ntiles; ++t, ++ai) {
    if (static_cast<int>(ai & 1u) != grp) continue;   // the other group's tile
    const uint32_t ab = ai % kAccBufs;
    if (!warp_wait(&ctl.acc_full[ab], (ai / kAccBufs) & 1u, P.wait_limit_ns, &ctl.abort))
      return false;
    tc_fence_after();
    float v[128];
    const uint32_t taddr = ctl.tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + ab * 128u;
#pragma unroll
    for (int c = 0; c < 4; ++c) tmem_ld32(taddr + 32u * c, v + 32 * c);
    tmem_wait_ld();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl.acc_empty[ab]);
    const int key0 = split * kSplitKeys + t * kTileKeys;
    if (key0 + kTileKeys - 1 > lim_all) {
#pragma unroll
      for (int j = 0; j < 128; ++j)
        if (key0 + j > lim) v[j] = -INFINITY;
    }
    float mx = v[0];
#pragma unroll
    for (int j = 1; j + 1 < 128; j += 2) mx = max3(mx, v[j], v[j + 1]);
    mx = fmaxf(mx, v[127]);
    const float mn = fmaxf(m, mx * alpha);
    if (mn != -INFINITY) {
      const float2 a2 = make_float2(alpha, alpha);
      const float2 nm2 = make_float2(-mn, -mn);
      float2 s0 = make_float2(0.f, 0.f), s1 = s0, s2 = s0, s3 = s0;
#pragma unroll
      for (int j = 0; j < 128; j += 8) {
        float2 x[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) x[k] = ffma2(make_float2(v[j + 2 * k], v[j + 2 * k + 1]), a2, nm2);
        s0 = fadd2(s0, make_float2(ex2(x[0].x), ex2(x[0].y)));
        s1 = fadd2(s1, make_float2(ex2(x[1].x), ex2(x[1].y)));
        s2 = fadd2(s2, make_float2(ex2(x[2].x), ex2(x[2].y)));
        s3 = fadd2(s3, make_float2(ex2(x[3].x), ex2(x[3].y)));
      }
      const float2 ss = fadd2(fadd2(s0, s1), fadd2(s2, s3));
      const float scale = (m == -INFINITY) ? 0.f : ex2(m - mn);
      Z = fmaf(Z, scale, ss.x + ss.y);
      m = mn;
    }
  }
  ctl.comb[slot][grp][row] = make_float2(m, Z);
  return true;
}

// ---------------------------------------------------------------- epilogue, phase 1

template <bool kFull>
__device__ __forceinline__ bool colstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, int split, uint32_t slot,
                                              uint32_t& ai) {
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int grp = (threadIdx.x - kEpiWarp0 * 32) >> 7;
  const int tl = quad * 32 + lane;         // key within the tile
  const int n = kFull ? kMaxRows : P.g.n_rows;
  const int nch = kFull ? 4 : (n + 31) / 32;
  const int W = P.g.window;
  const float alpha = P.alpha;
  const int ntiles = item_tiles(u.L, split);
  const float inv_n = 1.0f / static_cast<float>(n);
  const float inv_n1 = n > 1 ? 1.0f / static_cast<float>(n - 1) : 0.f;
  const float4* nb4 = reinterpret_cast<const float4*>(ctl.nbeta[slot]);
  const float2 a2 = make_float2(alpha, alpha);
  for (int t = 0; t < ntiles; ++t, ++ai) {
    if (static_cast<int>(ai & 1u) != grp) continue;
    const uint32_t ab = ai % kAccBufs;
    if (!warp_wait(&ctl.acc_full[ab], (ai / kAccBufs) & 1u, P.wait_limit_ns, &ctl.abort))
      return false;
    tc_fence_after();
    float v[128];
    const uint32_t taddr = ctl.tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + ab * 128u;
#pragma unroll
    for (int c = 0; c < 4; ++c)
      if (c < nch) tmem_ld32(taddr + 32u * c, v + 32 * c);
    tmem_wait_ld();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl.acc_empty[ab]);
    const int key = split * kSplitKeys + t * kTileKeys + tl;
    // A[r] = 2^(alpha*l - beta_r); rows that do not see this key (causal) get 0
#pragma unroll
    for (int r = 0; r < 128; r += 4) {
      if (kFull || r < n) {
        const float4 b = nb4[r >> 2];
        const float2 x0 = ffma2(make_float2(v[r], v[r + 1]), a2, make_float2(b.x, b.y));
        const float2 x1 = ffma2(make_float2(v[r + 2], v[r + 3]), a2, make_float2(b.z, b.w));
        v[r] = ex2(x0.x);
        v[r + 1] = ex2(x0.y);
        v[r + 2] = ex2(x1.x);
        v[r + 3] = ex2(x1.y);
      }
    }
    if (key > u.L - W) {
      const int rel = key - (u.L - W);
#pragma unroll
      for (int r = 0; r < 128; ++r)
        if ((kFull || r < n) && rel > ctl.roww[r]) v[r] = 0.f;
    }
    float mu, sigma;
    if (kFull) {
      float2 a0 = make_float2(0.f, 0.f), a1 = a0, a2s = a0, a3 = a0;
#pragma unroll
      for (int r = 0; r < 128; r += 8) {
        a0 = fadd2(a0, make_float2(v[r], v[r + 1]));
        a1 = fadd2(a1, make_float2(v[r + 2], v[r + 3]));
        a2s = fadd2(a2s, make_float2(v[r + 4], v[r + 5]));
        a3 = fadd2(a3, make_float2(v[r + 6], v[r + 7]));
      }
      const float2 as = fadd2(fadd2(a0, a1), fadd2(a2s, a3));
      mu = (as.x + as.y) * inv_n;
      const float2 nmu = make_float2(-mu, -mu);
      float2 q0 = make_float2(0.f, 0.f), q1 = q0, q2 = q0, q3 = q0;
#pragma unroll
      for (int r = 0; r < 128; r += 8) {
        const float2 d0 = fadd2(make_float2(v[r], v[r + 1]), nmu);
        const float2 d1 = fadd2(make_float2(v[r + 2], v[r + 3]), nmu);
        const float2 d2 = fadd2(make_float2(v[r + 4], v[r + 5]), nmu);
        const float2 d3 = fadd2(make_float2(v[r + 6], v[r + 7]), nmu);
        q0 = ffma2(d0, d0, q0);
        q1 = ffma2(d1, d1, q1);
        q2 = ffma2(d2, d2, q2);
        q3 = ffma2(d3, d3, q3);
      }
      const float2 qs = fadd2(fadd2(q0, q1), fadd2(q2, q3));
      sigma = sqrtf((qs.x + qs.y) * inv_n1);
    } else {
      float a = 0.f;
#pragma unroll
      for (int r = 0; r < 128; ++r)
        if (r < n) a += v[r];
      mu = a * inv_n;
      float q = 0.f;
#pragma unroll
      for (int r = 0; r < 128; ++r)
        if (r < n) {
          const float d = v[r] - mu;
          q = fmaf(d, d, q);
        }
      sigma = sqrtf(q * inv_n1);
    }
    if (key < u.L) {
      __stcs(&P.mu[u.mu_off + key], mu);
      __stcs(&P.sigma[u.mu_off + key], sigma);
    }
  }
  return true;
}

// ---------------------------------------------------------------- sync warp

// Phase-0 item: merge the two groups' (m, Z) per row, publish them, count the item,
// and if it is the unit's last, merge all of the unit's items into beta.
__device__ __forceinline__ bool sync_rowstats(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, int64_t p, uint32_t slot) {
  const int lane = threadIdx.x & 31;
  const int n = P.g.n_rows;
  float2 mz[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = lane + 32 * k;
    mz[k] = merge_mz(ctl.comb[slot][0][row], ctl.comb[slot][1][row]);
  }
  // the slot's shared data is in registers: hand the slot back to the producer
  __syncwarp();
  if (lane == 0) mbar_arrive(&ctl.item_empty[slot]);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = lane + 32 * k;
    if (row < n) P.partial[p * kMaxRows + row] = mz[k];
  }
  __threadfence();
  __syncwarp();
  int last = 0;
  if (lane == 0 && !(P.fault == 1 && u.unit == 0)) {
    const uint32_t old = atomicAdd(&P.counts[u.unit], 1u);
    last = (old == static_cast<uint32_t>(u.splits - 1));
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (last) {
    __threadfence();
    float2 acc[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) acc[k] = make_float2(-INFINITY, 0.f);
    for (int s0 = 0; s0 < u.splits; s0 += 8) {
      float2 pz[4][8];
#pragma unroll
      for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int row = lane + 32 * k;
          pz[k][j] = (s0 + j < u.splits && row < n)
                         ? __ldcg(&P.partial[(u.item0 + s0 + j) * kMaxRows + row])
                         : make_float2(-INFINITY, 0.f);
        }
#pragma unroll
      for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[k] = merge_mz(acc[k], pz[k][j]);
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int row = lane + 32 * k;
      if (row < n) {
        // one 64-bit store: a reader sees either the cleared word or (beta, 1)
        const float b = acc[k].x + lg2(acc[k].y);
        const unsigned long long word =
            (1ull << 32) | static_cast<unsigned long long>(__float_as_uint(b));
        __stcg(&P.beta[u.unit * kMaxRows + row], word);
      }
    }
    __threadfence();
    __syncwarp();
    if (lane == 0) st_release_gpu(&P.done[u.unit], 1u);   // hint for the producers
  }
  return true;
}

// Phase-1 item: wait for the unit's merged statistics and stage -beta. Each row's
// normaliser carries its own ready tag, so one round of loads both checks and
// fetches it.
__device__ __forceinline__ bool sync_colstats(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, uint32_t slot) {
  const int lane = threadIdx.x & 31;
  const int n = P.g.n_rows;
  const int r0 = 4 * lane;
  const uint64_t deadline = global_timer_ns() + P.wait_limit_ns;
  const volatile uint32_t* errw = P.err;
  uint32_t ns = 32;
  unsigned long long w[4];
  for (;;) {
#pragma unroll
    for (int k = 0; k < 4; ++k)
      w[k] = (r0 + k < n) ? __ldcg(&P.beta[u.unit * kMaxRows + r0 + k]) : (1ull << 32);
    bool ready = true;
#pragma unroll
    for (int k = 0; k < 4; ++k) ready = ready && (w[k] >> 32) != 0ull;
    if (__all_sync(0xffffffffu, ready)) break;
    int give_up = 0;
    if (lane == 0) give_up = (*errw != 0u || ctl.abort || global_timer_ns() > deadline) ? 1 : 0;
    if (__shfl_sync(0xffffffffu, give_up, 0)) return false;
    __nanosleep(ns);
    if (ns < 512) ns *= 2;
  }
  float4 b;
  b.x = r0 + 0 < n ? -__uint_as_float(static_cast<uint32_t>(w[0])) : -INFINITY;
  b.y = r0 + 1 < n ? -__uint_as_float(static_cast<uint32_t>(w[1])) : -INFINITY;
  b.z = r0 + 2 < n ? -__uint_as_float(static_cast<uint32_t>(w[2])) : -INFINITY;
  b.w = r0 + 3 < n ? -__uint_as_float(static_cast<uint32_t>(w[3])) : -INFINITY;
  reinterpret_cast<float4*>(ctl.nbeta[slot])[lane] = b;
  return true;
}

// ---------------------------------------------------------------- kernel

template <bool kFull>
__global__ void __launch_bounds__(kThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ ScoreParams P) {
  __shared__ ScoreCtl ctl;
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* qbuf = tiles;                             // kQBufs x 32 KB
  uint8_t* kbuf = tiles + kQBufs * kTileBytes;       // kKStages x 32 KB

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t n1 = P.g.n_items;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kQBufs; ++i) { mbar_init(&ctl.q_full[i], 1); mbar_init(&ctl.q_empty[i], 1); }
    for (int i = 0; i < kKStages; ++i) { mbar_init(&ctl.k_full[i], 1); mbar_init(&ctl.k_empty[i], 1); }
    for (int i = 0; i < kAccBufs; ++i) { mbar_init(&ctl.acc_full[i], 1); mbar_init(&ctl.acc_empty[i], 4); }
    for (int i = 0; i < kItemSlots; ++i) {
      mbar_init(&ctl.item_full[i], 1);
      mbar_init(&ctl.item_empty[i], 2 + kEpiWarps);   // MMA + sync + epilogue warps
      mbar_init(&ctl.pub_full[i], kEpiWarps);
      mbar_init(&ctl.beta_full[i], 1);
    }
    ctl.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&tm_q);
    prefetch_tensormap(&tm_k);
  }
  if (threadIdx.x < kMaxRows) ctl.roww[threadIdx.x] = threadIdx.x % P.g.window;
  if (warp == 1) {
    tmem_alloc(&ctl.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t it = 0, qi = 0, ki = 0;
      int q_used[kQBufs] = {0, 0}, k_used[kKStages] = {0, 0, 0, 0};
      uint32_t q_last[kQBufs] = {0, 0}, k_last[kKStages] = {0, 0, 0, 0};
      const uint64_t pol_keep = l2_policy_evict_last();
      const uint64_t pol_drop = l2_policy_evict_first();
      bool ok = true;
      // Row items are claimed one ahead. Column items are claimed only when the unit
      // at the head of the column queue is ready: the head index and its unit's done
      // flag are polled with relaxed loads whose values are used one item later. A
      // claim that raced past the ready front is held until its unit is ready.
      const volatile uint32_t* errw = P.err;
      int s2;
      int64_t p1 = atomicAdd(P.claim1, 1u);
      int64_t held = -1;                               // claimed, not yet ready
      int64_t head = 0;                                // queue head the flag refers to
      uint32_t head_ready = 0;                         // done flag of head's unit
      int64_t peek = 0;                                // newest peek of the queue head
      uint32_t held_ready = 0;
      for (;;) {
        Claim cl;
        bool have = false;
        if (ctl.abort) {
          have = false;
        } else if (held >= 0 && held_ready) {
          cl.phase = 1;
          cl.p = held;
          have = true;
          held = -1;
        } else if (held < 0 && head < n1 && head_ready) {
          const int64_t q = atomicAdd(P.claim2, 1u);
          if (q < n1) {
            if (item_unit(P.g, q, &s2) == item_unit(P.g, head, &s2)) {
              cl.phase = 1;
              cl.p = q;
              have = true;
            } else {
              held = q;
              held_ready = 0;
            }
          }
        }
        if (!have && !ctl.abort && p1 < n1) {
          cl.phase = 0;
          cl.p = p1;
          have = true;
          p1 = atomicAdd(P.claim1, 1u);
        }
        if (!have && !ctl.abort) {
          // no row work left: wait (bounded) for column work to become ready
          const int64_t h = ld_volatile_u32(P.claim2);
          if (held < 0 && h >= n1) {
            have = false;                              // all work is claimed: finish
          } else {
            const uint64_t deadline = global_timer_ns() + P.wait_limit_ns;
            uint32_t ns = 64;
            bool ready = false;
            for (;;) {
              const int64_t x = held >= 0 ? held : static_cast<int64_t>(ld_volatile_u32(P.claim2));
              if (x >= n1) break;
              if (ld_volatile_u32(&P.done[item_unit(P.g, x, &s2)])) {
                ready = true;
                break;
              }
              if (*errw != 0u || ctl.abort || global_timer_ns() > deadline) break;
              __nanosleep(ns);
              if (ns < 1024) ns *= 2;
            }
            if (held >= 0) {
              if (!ready) {
                ok = false;
                break;
              }
              held_ready = 1;
            } else {
              if (!ready && ld_volatile_u32(P.claim2) < n1) {
                ok = false;
                break;
              }
              head = ld_volatile_u32(P.claim2);
              peek = head;
              head_ready = ready ? 1u : 0u;
            }
            continue;
          }
        }
        // refresh the polls, consumed at the next decision: the done flag of the
        // head peeked last time, and an independent new peek of the head
        if (held >= 0) {
          held_ready = ld_volatile_u32(&P.done[item_unit(P.g, held, &s2)]);
        } else {
          head = peek;
          head_ready = head < n1 ? ld_volatile_u32(&P.done[item_unit(P.g, head, &s2)]) : 0u;
          peek = ld_volatile_u32(P.claim2);
        }
        const uint32_t slot = it % kItemSlots;
        if (!mbar_wait(&ctl.item_empty[slot], ((it / kItemSlots) & 1u) ^ 1u,
                       global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        ctl.item_ring[slot] = have ? encode_claim(cl.phase, cl.p) : -1;
        mbar_arrive(&ctl.item_full[slot]);
        ++it;
        if (!have) break;
        int split;
        const UnitInfo u = unit_info(P.g, item_unit(P.g, cl.p, &split));
        const uint32_t qb = qi % kQBufs;
        if (!mbar_wait(&ctl.q_empty[qb], ((qi / kQBufs) & 1u) ^ 1u,
                       global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&ctl.q_full[qb], kTileBytes);
        tma_load_2d(qbuf + qb * kTileBytes, &tm_q, 0, static_cast<int32_t>(u.q_row0), &ctl.q_full[qb]);
        tma_load_2d(qbuf + qb * kTileBytes + kHalfBytes, &tm_q, 64, static_cast<int32_t>(u.q_row0),
                    &ctl.q_full[qb]);
        q_used[qb] = 1;
        q_last[qb] = (qi / kQBufs) & 1u;
        ++qi;
        const int ntiles = item_tiles(u.L, split);
        const uint64_t pol = cl.phase == 0 ? pol_keep : pol_drop;
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t ks = ki % kKStages;
          if (!mbar_wait(&ctl.k_empty[ks], ((ki / kKStages) & 1u) ^ 1u,
                         global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
            ok = false;
            break;
          }
          const int32_t y = static_cast<int32_t>(u.k_row0 + split * kSplitKeys + t * kTileKeys);
          mbar_arrive_expect_tx(&ctl.k_full[ks], kTileBytes);
          tma_load_2d_hint(kbuf + ks * kTileBytes, &tm_k, 0, y, &ctl.k_full[ks], pol);
          tma_load_2d_hint(kbuf + ks * kTileBytes + kHalfBytes, &tm_k, 64, y, &ctl.k_full[ks], pol);
          k_used[ks] = 1;
          k_last[ks] = (ki / kKStages) & 1u;
          ++ki;
        }
        if (!ok) break;
      }
      if (!ok) set_error(P, ctl, 1u);
      // no bulk copy may still be writing shared memory when the CTA exits
      volatile int no_abort = 0;
      for (int i = 0; i < kQBufs; ++i)
        if (q_used[i]) mbar_wait(&ctl.q_full[i], q_last[i], global_timer_ns() + P.wait_limit_ns, &no_abort);
      for (int i = 0; i < kKStages; ++i)
        if (k_used[i]) mbar_wait(&ctl.k_full[i], k_last[i], global_timer_ns() + P.wait_limit_ns, &no_abort);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t it = 0, qi = 0, ki = 0, ai = 0;
      int issued = 0;
      uint32_t last_ab = 0, last_par = 0;
      const uint32_t qaddr = smem_u32(qbuf);
      const uint32_t kaddr = smem_u32(kbuf);
      bool ok = true;
      for (;;) {
        const uint32_t slot = it % kItemSlots;
        if (!mbar_wait(&ctl.item_full[slot], (it / kItemSlots) & 1u,
                       global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        const int64_t c = ctl.item_ring[slot];
        mbar_arrive(&ctl.item_empty[slot]);
        ++it;
        if (c < 0) break;
        const Claim cl = decode_claim(c);
        int split;
        const UnitInfo u = unit_info(P.g, item_unit(P.g, cl.p, &split));
        const uint32_t qb = qi % kQBufs;
        if (!mbar_wait(&ctl.q_full[qb], (qi / kQBufs) & 1u, global_timer_ns() + P.wait_limit_ns,
                       &ctl.abort)) {
          ok = false;
          break;
        }
        ++qi;
        const int ntiles = item_tiles(u.L, split);
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t ks = ki % kKStages;
          const uint32_t ab = ai % kAccBufs;
          if (!mbar_wait(&ctl.k_full[ks], (ki / kKStages) & 1u, global_timer_ns() + P.wait_limit_ns,
                         &ctl.abort) ||
              !mbar_wait(&ctl.acc_empty[ab], ((ai / kAccBufs) & 1u) ^ 1u,
                         global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = ctl.tmem_base + ab * 128u;
#pragma unroll
          for (int j = 0; j < kHeadDim / 16; ++j) {
            const uint32_t off = (j >> 2) * kHalfBytes + (j & 3) * 32u;
            const uint64_t qd = sw128_desc(qaddr + qb * kTileBytes + off);
            const uint64_t kd = sw128_desc(kaddr + ks * kTileBytes + off);
            if (cl.phase == 0)
              tc_mma_bf16(d_tmem, qd, kd, kIdesc, j > 0 ? 1u : 0u);
            else
              tc_mma_bf16(d_tmem, kd, qd, kIdesc, j > 0 ? 1u : 0u);
          }
          tc_commit(&ctl.k_empty[ks]);
          tc_commit(&ctl.acc_full[ab]);
          issued = 1;
          last_ab = ab;
          last_par = (ai / kAccBufs) & 1u;
          ++ki;
          ++ai;
        }
        if (!ok) break;
        tc_commit(&ctl.q_empty[qb]);
      }
      if (!ok) set_error(P, ctl, 1u);
      // the MMAs must have finished before TMEM is released
      volatile int no_abort = 0;
      if (issued)
        mbar_wait(&ctl.acc_full[last_ab], last_par, global_timer_ns() + P.wait_limit_ns, &no_abort);
    }
  } else if (warp == kSyncWarp) {
    // ------------------------------------------------------------ sync warp
    uint32_t it = 0;
    for (;;) {
      const uint32_t slot = it % kItemSlots;
      const uint32_t par = (it / kItemSlots) & 1u;
      if (!warp_wait(&ctl.item_full[slot], par, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const int64_t c = ctl.item_ring[slot];
      if (c < 0) break;
      const Claim cl = decode_claim(c);
      int split;
      const UnitInfo u = unit_info(P.g, item_unit(P.g, cl.p, &split));
      bool ok;
      if (cl.phase == 0) {
        if (lane == 0) mbar_arrive(&ctl.beta_full[slot]);      // nothing to stage
        ok = warp_wait(&ctl.pub_full[slot], par, P.wait_limit_ns, &ctl.abort) &&
             sync_rowstats(P, ctl, u, cl.p, slot);            // hands the slot back early
      } else {
        ok = sync_colstats(P, ctl, u, slot);
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&ctl.beta_full[slot]);
          mbar_arrive(&ctl.item_empty[slot]);
        }
      }
      if (!ok) {
        set_error(P, ctl, 1u);
        break;
      }
      ++it;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    uint32_t it = 0, ai = 0;
    for (;;) {
      const uint32_t slot = it % kItemSlots;
      const uint32_t par = (it / kItemSlots) & 1u;
      if (!warp_wait(&ctl.item_full[slot], par, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const int64_t c = ctl.item_ring[slot];
      if (c < 0) break;
      const Claim cl = decode_claim(c);
      int split;
      const UnitInfo u = unit_info(P.g, item_unit(P.g, cl.p, &split));
      bool ok;
      if (cl.phase == 0) {
        ok = rowstats_item<kFull>(P, ctl, u, split, slot, ai);
      } else {
        ok = warp_wait(&ctl.beta_full[slot], par, P.wait_limit_ns, &ctl.abort) &&
             colstats_item<kFull>(P, ctl, u, split, slot, ai);
      }
      if (!ok) {
        set_error(P, ctl, 1u);
        break;
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&ctl.pub_full[slot]);
        mbar_arrive(&ctl.item_empty[slot]);
      }
      ++it;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(ctl.tmem_base, kTmemCols);
  }
}

}  // namespace

cudaError_t launch_score(const kve_plan& plan, const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                         const ScoreParams& p, int num_sms, cudaStream_t stream) {
  const bool full = plan.geo.n_rows == kMaxRows;
  auto* fn = full ? score_kernel<true> : score_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kDynSmem));
  if (e != cudaSuccess) return e;
  const int64_t items = p.g.n_items;
  const int grid = static_cast<int>(items < num_sms ? items : num_sms);
  fn<<<grid, kThreads, kDynSmem, stream>>>(tm_q, tm_k, p);
  return cudaGetLastError();
}

}  // namespace kve
