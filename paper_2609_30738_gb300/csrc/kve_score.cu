// Window-score kernel: steps 1-2 of the eviction step (Section 3.1, Eq. 1, Eq. 3).
//
// For every unit (request, layer, KV head) the n = G*W window rows attend to the
// L prefix keys through a causal softmax; mu_i and sigma_i are the mean and the
// sample standard deviation of A[., i] over the n rows.
//
// Work is cut into items of up to 512 keys (4 tiles of 128). Each item runs in one
// of two phases on a persistent, warp-specialised CTA:
//   phase 0 (row statistics):   D[row][key] = Q K^T on tcgen05 (rows on TMEM lanes);
//                               each epilogue thread owns one row and keeps the
//                               running max m and sum Z = sum 2^(alpha*l - m) of its
//                               row over the item's keys, then publishes (m, Z).
//                               The last item of a unit to publish merges all of
//                               them into beta_r = log2 of the row's softmax
//                               normaliser and raises the unit's ready flag.
//   phase 1 (column statistics): D[key][row] = K Q^T (keys on TMEM lanes); each
//                               epilogue thread owns one key, forms
//                               A = 2^(alpha*l - beta_r) for its n rows and reduces
//                               them to mu and sigma in registers (two passes).
// Items are claimed in a global order in which every phase-0 item of a unit comes
// before any phase-1 item of it, and phase-1 items trail phase-0 items by `lag`
// items so that their K tiles are still in L2. A CTA processes its claims in
// order, so a phase-1 item only ever waits for phase-0 items claimed before it;
// the wait is bounded and reports KVE_ETIMEOUT instead of hanging.
//
// Roles: warp 0 claims items and issues TMA loads, warp 1 owns TMEM and issues
// the MMAs, warps 2-5 run the epilogue (warp w reads TMEM lanes 32*(w%4)..+31).
#include "kve_internal.h"
#include "kve_ptx.cuh"

namespace kve {
namespace {

constexpr int kThreads = 192;
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
  uint64_t epi_bar;
  int64_t item_ring[kItemSlots];
  uint32_t tmem_base;
  volatile int abort;
  volatile int is_last;
  float nbeta[kMaxRows];
  int32_t roww[kMaxRows];
};

struct Claim {
  int phase;
  int64_t p;
};

__device__ __forceinline__ Claim decode_claim(int64_t c, int64_t n1, int64_t lag) {
  Claim k;
  if (c < lag) {
    k.phase = 0;
    k.p = c;
    return k;
  }
  const int64_t j = c - lag;
  const int64_t inter = 2 * (n1 - lag);
  if (j < inter) {
    k.phase = static_cast<int>(j & 1);
    k.p = (j & 1) ? (j >> 1) : lag + (j >> 1);
  } else {
    k.phase = 1;
    k.p = j - (n1 - lag);
  }
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

// Bounded barrier among the 4 epilogue warps (an mbarrier with 4 arrivals).
__device__ __forceinline__ bool epi_sync(ScoreCtl& ctl, uint32_t& phase, uint64_t limit) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&ctl.epi_bar);
  const bool ok = warp_wait(&ctl.epi_bar, phase, limit, &ctl.abort);
  phase ^= 1u;
  return ok;
}

// ---------------------------------------------------------------- epilogue, phase 0

template <bool kFull>
__device__ __forceinline__ bool rowstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, int split, int64_t p,
                                              uint32_t& ai, uint32_t& epi_phase) {
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int row = quad * 32 + lane;
  const int n = P.g.n_rows;
  const int W = P.g.window;
  const int lim_all = u.L - W;                 // keys <= lim_all are seen by every row
  const int lim = u.L - W + ctl.roww[row];     // last key this row sees
  const int ntiles = item_tiles(u.L, split);
  const float alpha = P.alpha;
  float m = -INFINITY, Z = 0.f;
  for (int t = 0; t < ntiles; ++t) {
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
    ++ai;
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
      float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
      for (int j = 0; j < 128; j += 4) {
        s0 += ex2(fmaf(v[j + 0], alpha, -mn));
        s1 += ex2(fmaf(v[j + 1], alpha, -mn));
        s2 += ex2(fmaf(v[j + 2], alpha, -mn));
        s3 += ex2(fmaf(v[j + 3], alpha, -mn));
      }
      const float scale = (m == -INFINITY) ? 0.f : ex2(m - mn);
      Z = fmaf(Z, scale, (s0 + s1) + (s2 + s3));
      m = mn;
    }
  }
  if (kFull || row < n) {
    P.partial[p * kMaxRows + row] = make_float2(m, Z);
  }
  __threadfence();
  if (!epi_sync(ctl, epi_phase, P.wait_limit_ns)) return false;
  if (threadIdx.x == 64) {
    int last = 0;
    if (!(P.fault == 1 && u.unit == 0)) {
      const uint32_t old = atomicAdd(&P.counts[u.unit], 1u);
      last = (old == static_cast<uint32_t>(u.splits - 1));
    }
    ctl.is_last = last;
  }
  if (!epi_sync(ctl, epi_phase, P.wait_limit_ns)) return false;
  if (ctl.is_last) {
    __threadfence();
    if (kFull || row < n) {
      float mg = -INFINITY;
      for (int s = 0; s < u.splits; ++s)
        mg = fmaxf(mg, __ldcg(&P.partial[(u.item0 + s) * kMaxRows + row]).x);
      float zg = 0.f;
      for (int s = 0; s < u.splits; ++s) {
        const float2 pz = __ldcg(&P.partial[(u.item0 + s) * kMaxRows + row]);
        if (pz.x != -INFINITY) zg = fmaf(pz.y, ex2(pz.x - mg), zg);
      }
      __stcg(&P.beta[u.unit * kMaxRows + row], mg + lg2(zg));
    }
    __threadfence();
    if (!epi_sync(ctl, epi_phase, P.wait_limit_ns)) return false;
    if (threadIdx.x == 64) st_release_gpu(&P.flags[u.unit], 1u);
  }
  return true;
}

// ---------------------------------------------------------------- epilogue, phase 1

template <bool kFull>
__device__ __forceinline__ bool colstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const UnitInfo& u, int split, uint32_t& ai,
                                              uint32_t& epi_phase) {
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int tl = quad * 32 + lane;         // key within the tile
  const int n = kFull ? kMaxRows : P.g.n_rows;
  const int nch = kFull ? 4 : (n + 31) / 32;
  const int W = P.g.window;
  const float alpha = P.alpha;
  // wait for the unit's merged row statistics
  if (threadIdx.x == 64) {
    const uint64_t deadline = global_timer_ns() + P.wait_limit_ns;
    const volatile uint32_t* errw = P.err;
    uint32_t ns = 32;
    while (ld_acquire_gpu(&P.flags[u.unit]) == 0u) {
      if (*errw != 0u || global_timer_ns() > deadline) {
        set_error(P, ctl, 1u);
        break;
      }
      __nanosleep(ns);
      if (ns < 1024) ns *= 2;
    }
  }
  if (!epi_sync(ctl, epi_phase, P.wait_limit_ns)) return false;
  if (ctl.abort) return false;
  ctl.nbeta[tl] = (tl < P.g.n_rows) ? -__ldcg(&P.beta[u.unit * kMaxRows + tl]) : -INFINITY;
  if (!epi_sync(ctl, epi_phase, P.wait_limit_ns)) return false;

  const int ntiles = item_tiles(u.L, split);
  const float inv_n = 1.0f / static_cast<float>(n);
  const float inv_n1 = n > 1 ? 1.0f / static_cast<float>(n - 1) : 0.f;
  for (int t = 0; t < ntiles; ++t) {
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
    ++ai;
    const int key = split * kSplitKeys + t * kTileKeys + tl;
    // A[r] = 2^(alpha*l - beta_r); rows that do not see this key (causal) get 0
#pragma unroll
    for (int r = 0; r < 128; ++r) {
      if (kFull || r < n) v[r] = ex2(fmaf(v[r], alpha, ctl.nbeta[r]));
    }
    if (key > u.L - W) {
      const int rel = key - (u.L - W);
#pragma unroll
      for (int r = 0; r < 128; ++r)
        if ((kFull || r < n) && rel > ctl.roww[r]) v[r] = 0.f;
    }
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
    for (int r = 0; r < 128; r += 4) {
      if (kFull || r + 0 < n) a0 += v[r + 0];
      if (kFull || r + 1 < n) a1 += v[r + 1];
      if (kFull || r + 2 < n) a2 += v[r + 2];
      if (kFull || r + 3 < n) a3 += v[r + 3];
    }
    const float mu = ((a0 + a1) + (a2 + a3)) * inv_n;
    float q0 = 0.f, q1 = 0.f, q2 = 0.f, q3 = 0.f;
#pragma unroll
    for (int r = 0; r < 128; r += 4) {
      float d;
      if (kFull || r + 0 < n) { d = v[r + 0] - mu; q0 = fmaf(d, d, q0); }
      if (kFull || r + 1 < n) { d = v[r + 1] - mu; q1 = fmaf(d, d, q1); }
      if (kFull || r + 2 < n) { d = v[r + 2] - mu; q2 = fmaf(d, d, q2); }
      if (kFull || r + 3 < n) { d = v[r + 3] - mu; q3 = fmaf(d, d, q3); }
    }
    const float sigma = sqrtf(((q0 + q1) + (q2 + q3)) * inv_n1);
    if (key < u.L) {
      __stcs(&P.mu[u.mu_off + key], mu);
      __stcs(&P.sigma[u.mu_off + key], sigma);
    }
  }
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
  const int64_t total_claims = 2 * n1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kQBufs; ++i) { mbar_init(&ctl.q_full[i], 1); mbar_init(&ctl.q_empty[i], 1); }
    for (int i = 0; i < kKStages; ++i) { mbar_init(&ctl.k_full[i], 1); mbar_init(&ctl.k_empty[i], 1); }
    for (int i = 0; i < kAccBufs; ++i) { mbar_init(&ctl.acc_full[i], 1); mbar_init(&ctl.acc_empty[i], 4); }
    for (int i = 0; i < kItemSlots; ++i) { mbar_init(&ctl.item_full[i], 1); mbar_init(&ctl.item_empty[i], 5); }
    mbar_init(&ctl.epi_bar, 4);
    ctl.abort = 0;
    ctl.is_last = 0;
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
      for (;;) {
        int64_t c = ctl.abort ? total_claims : static_cast<int64_t>(atomicAdd(P.claim, 1u));
        if (c > total_claims) c = total_claims;
        const uint32_t slot = it % kItemSlots;
        if (!mbar_wait(&ctl.item_empty[slot], ((it / kItemSlots) & 1u) ^ 1u,
                       global_timer_ns() + P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        ctl.item_ring[slot] = (c >= total_claims) ? -1 : c;
        mbar_arrive(&ctl.item_full[slot]);
        ++it;
        if (c >= total_claims) break;
        const Claim cl = decode_claim(c, n1, P.lag);
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
        const Claim cl = decode_claim(c, n1, P.lag);
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
  } else {
    // ------------------------------------------------------------ epilogue
    uint32_t it = 0, ai = 0, epi_phase = 0;
    for (;;) {
      const uint32_t slot = it % kItemSlots;
      if (!warp_wait(&ctl.item_full[slot], (it / kItemSlots) & 1u, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const int64_t c = ctl.item_ring[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.item_empty[slot]);
      ++it;
      if (c < 0) break;
      const Claim cl = decode_claim(c, n1, P.lag);
      int split;
      const UnitInfo u = unit_info(P.g, item_unit(P.g, cl.p, &split));
      const bool ok = (cl.phase == 0)
                          ? rowstats_item<kFull>(P, ctl, u, split, cl.p, ai, epi_phase)
                          : colstats_item<kFull>(P, ctl, u, split, ai, epi_phase);
      if (!ok) {
        set_error(P, ctl, 1u);
        break;
      }
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
  const int64_t claims = 2 * p.g.n_items;
  const int grid = static_cast<int>(claims < num_sms ? claims : num_sms);
  fn<<<grid, kThreads, kDynSmem, stream>>>(tm_q, tm_k, p);
  return cudaGetLastError();
}

}  // namespace kve
