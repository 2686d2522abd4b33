// Window-score kernel: steps 1-2 of the eviction step (Section 3.1, Eq. 1, Eq. 3).
//
// For every unit (request, layer, KV head) the n = G*W window rows attend to the
// L prefix keys through a causal softmax; mu_i and sigma_i are the mean and the
// sample standard deviation of A[., i] over the n rows.
//
// Work is cut into items of at most kSplitTiles tiles of 128 keys. Each item runs in
// one of two phases on a persistent, warp-specialised CTA:
//   phase 0 (row statistics):   D[row][key] = Q K^T on tcgen05 (rows on TMEM lanes);
//                               each epilogue thread owns one row and keeps the
//                               running max m and sum Z = sum 2^(alpha*l - m) of its
//                               row; the item's (m, Z) per row are published, and
//                               the last item of a unit to publish merges them into
//                               beta_r = log2 of the row's softmax normaliser.
//   phase 1 (column statistics): D[key][row] = K Q^T (keys on TMEM lanes); each
//                               epilogue thread owns one key, forms
//                               A = 2^(alpha*l - beta_r) for its n rows and reduces
//                               them to mu and sigma in registers (sums and sums of
//                               squares; two passes where sigma/mu is small).
// The schedule is static. CTA c owns items c, c + G, c + 2G, ... (G CTAs, all
// resident: the launch is cooperative), so round j is items [jG, (j+1)G) and a
// unit's items run side by side in one round (the host picks the items per unit so
// that rounds hold whole units). A CTA runs the phase-0 pass of its round-j item,
// then the phase-1 pass of its round-(j - lag) item. A unit's items span at most
// lag - 1 rounds (the host computes lag from the geometry), so every phase-1 item
// waits only on phase-0 work that comes earlier in every CTA's sequence: there is
// no circular wait. Between the two passes over an item's K tiles the GPU streams
// about one round of other tiles, far less than L2 holds, so the phase-1 pass
// reads its tiles from L2. Every cross-CTA wait is bounded and a timeout is
// reported as KVE_ETIMEOUT.
//
// Roles: warp 0 walks the item sequence and issues TMA loads; warp 1 owns TMEM and
// issues the MMAs; warp 2 (sync) does the cross-CTA work in sequence order -- it
// publishes the row statistics of phase-0 items and stages -beta of phase-1 items
// in shared memory ahead of use; when a phase-0 item is the last of its unit to
// arrive, warp 2 hands the unit to warp 3 (merge), which folds the unit's partials
// into beta off the sequence's critical path; warps 4-11 run the epilogue in two
// groups of four (warp w reads TMEM lanes 32*(w%4)..+31), the groups taking
// alternate tiles. The epilogue warps never touch global synchronisation; they only
// compute, write shared memory and arrive on mbarriers.
#include <cstddef>

#include "kve_internal.h"
#include "kve_ptx.cuh"

namespace kve {
namespace {

constexpr int kThreads = 384;
// Control warps come first: a scheduler that favours older warps then serves the
// single-thread producer and MMA issuer and the latency-bound sync and merge warps
// ahead of the throughput-bound epilogue.
constexpr int kSyncWarp = 2;
constexpr int kMergeWarp = 3;
constexpr int kEpiWarp0 = 4;
constexpr int kEpiWarps = 8;
constexpr int kMergeSlots = 4;
constexpr int kMaxQBufs = 2;
constexpr int kItemSlots = 4;
constexpr uint32_t kTileBytes = 128 * kHeadDim * 2;   // 32 KB: 128 rows x 128 bf16
constexpr uint32_t kHalfBytes = kTileBytes / 2;       // one 64-element (128 B) column block
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);
// O^T += V^T P^T with both operands MN-major (128-byte swizzle): instruction descriptor
// with the A and B transpose bits, and the operand strides of a [128][128] bf16 tile in
// two 64-column halves (16 KB apart along MN, 8-row groups 1 KB apart along K)
constexpr uint32_t kIdescMN = kIdesc | (1u << 15) | (1u << 16);
constexpr uint32_t kMNLbo = kHalfBytes;
constexpr uint32_t kMNSbo = 1024;

// Pipeline depths of the two variants. The plain kernel: 2 Q buffers, 3 K stages, 4
// score accumulators, partials merged 40 per bulk copy. With the window output (kAttn)
// the column pass also streams V and accumulates O^T on the tensor cores: a column
// tile's K stage holds its probabilities P^T until the O^T MMA has read them, so the
// shared memory goes to 3 K stages and 2 V stages with a single Q buffer and a merge
// buffer for 16 partials (measured: 1.84 ms per call at L = 32768 against 1.97 ms with
// 2 Q buffers, 2 K stages and 8 partials); 3 score accumulators and the O^T accumulator
// in TMEM columns 384..511.
template <bool kAttn>
struct Cfg {
  static constexpr int kQBufs = kAttn ? 1 : 2;
  static constexpr int kKStages = 3;
  static constexpr int kVStages = kAttn ? 2 : 0;
  static constexpr int kAccBufs = kAttn ? 3 : 4;
  static constexpr int kMergeBatch = kAttn ? 16 : 40;   // partials per bulk copy (1 KB each)
  static constexpr size_t kMergeBytes = static_cast<size_t>(kMergeBatch) * kMaxRows * sizeof(float2);
  static constexpr size_t kDynSmem = (kQBufs + kKStages + kVStages) * kTileBytes + kMergeBytes + 1024;
};
constexpr int kMaxKStages = 3;
static_assert(Cfg<false>::kKStages <= kMaxKStages && Cfg<true>::kKStages <= kMaxKStages, "K stage arrays");
static_assert(Cfg<true>::kVStages <= 2, "V stage arrays");
static_assert(Cfg<false>::kQBufs <= kMaxQBufs && Cfg<true>::kQBufs <= kMaxQBufs, "Q buffer arrays");
constexpr int kMaxAccBufs = 4;
constexpr uint32_t kOCol = 384;   // TMEM column of the O^T accumulator (window output)

// One pass over one item, as the producer derives it once from the item index and
// hands it to the other roles through the item ring (p = -1 ends the work).
struct ItemDesc {
  int64_t p;         // item index
  int64_t unit;
  int64_t mu_off;    // first mu/sigma element of the unit
  int64_t item0;     // first item of the unit
  int32_t phase;     // 0: row statistics, 1: column statistics
  int32_t tile0;     // first tile of the item within the unit
  int32_t ntiles;
  int32_t L;         // prefix length of the unit
  int32_t splits;    // items of the unit
  int32_t tok0;      // K tile coordinates: the unit's first token, KV head and layer
  int32_t kvh;
  int32_t layer;
};

struct Claim {
  int phase;
  int64_t p;
};

struct MergeJob {
  int64_t unit;      // -1: no more units
  int64_t item0;
  int32_t splits;
  int32_t pad;
};

struct ScoreCtl {
  uint64_t q_full[kMaxQBufs], q_empty[kMaxQBufs];
  uint64_t k_full[kMaxKStages], k_empty[kMaxKStages];
  uint64_t acc_full[kMaxAccBufs], acc_empty[kMaxAccBufs];
  // window output only: V stages, P^T written into a K stage, the O^T accumulator
  uint64_t v_full[2], v_empty[2];
  uint64_t p_full[kMaxKStages];     // epilogue -> MMA: P^T of the tile in K stage s is written
  uint64_t o_full, o_empty;         // MMA -> epilogue group 0 -> MMA, once per column item
  uint64_t item_full[kItemSlots], item_empty[kItemSlots];
  uint64_t pub_full[kItemSlots];    // epilogue -> sync warp, once per item
  uint64_t beta_full[kItemSlots];   // sync warp -> epilogue, once per item
  uint64_t merge_full[kMergeSlots], merge_empty[kMergeSlots];   // sync warp <-> merge warp
  ItemDesc item_ring[kItemSlots];   // written by the producer, read by every role
  MergeJob merge_job[kMergeSlots];  // unit to merge; unit -1 ends the merge warp
  uint64_t merge_bar;               // bulk copies of partials
  uint32_t tmem_base;
  volatile int abort;
  int32_t roww[kMaxRows];                            // r % W
  float rowm[kMaxRows];                              // 1 for rows r < n, else 0
  alignas(16) float2 comb[kItemSlots][2][kMaxRows];  // per group (m, Z) of a row item
  alignas(16) float nbeta[kItemSlots][kMaxRows];     // kColScale - beta of a column item
};
static_assert(offsetof(ScoreCtl, nbeta) % 16 == 0, "nbeta is read with 16-byte loads");
static_assert(offsetof(ScoreCtl, comb) % 16 == 0, "comb holds float2");


__device__ __forceinline__ void set_error(const ScoreParams& P, ScoreCtl& ctl, uint32_t code) {
  atomicOr(P.err, code);
  ctl.abort = 1;
}

// Bounded wait whose outcome is the same for every lane of the warp, so that a
// warp never splits in front of a .sync.aligned instruction.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit,
                                          volatile int* abort) {
  const bool ok = mbar_wait(bar, parity, limit, abort);
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

template <bool kFull, bool kAttn>
__device__ __forceinline__ bool rowstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const ItemDesc& d, uint32_t slot, uint32_t& ai) {
  constexpr int kAccBufs = Cfg<kAttn>::kAccBufs;
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int grp = (threadIdx.x - kEpiWarp0 * 32) >> 7;   // 0 or 1
  const int row = quad * 32 + lane;
  const int W = P.g.window;
  const int lim_all = d.L - W;                 // keys <= lim_all are seen by every row
  const int lim = d.L - W + ctl.roww[row];     // last key this row sees
  const int tile0 = d.tile0, ntiles = d.ntiles;
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
    const int key0 = (tile0 + t) * kTileKeys;
    if (key0 + kTileKeys - 1 > lim_all) {
#pragma unroll
      for (int j = 0; j < 128; ++j)
        if (key0 + j > lim) v[j] = -INFINITY;
    }
    float q0 = v[0], q1 = v[1], q2 = v[2], q3 = v[3];
#pragma unroll
    for (int j = 4; j < 124; j += 8) {
      q0 = max3(q0, v[j], v[j + 1]);
      q1 = max3(q1, v[j + 2], v[j + 3]);
      q2 = max3(q2, v[j + 4], v[j + 5]);
      q3 = max3(q3, v[j + 6], v[j + 7]);
    }
    q0 = max3(q0, v[124], v[125]);
    q1 = max3(q1, v[126], v[127]);
    const float mx = fmaxf(fmaxf(q0, q1), fmaxf(q2, q3));
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

// Column statistics are formed on A' = 2^kColScale * A (the staged normaliser is
// -beta_r + kColScale): squares of A' stay normal down to A ~ 2^-103, and every sum
// below stays far from fp32 overflow (A' <= 2^40, n <= 128).
constexpr float kColScale = 40.f;
constexpr float kColUnscale = 1.0f / 1099511627776.0f;   // 2^-40
constexpr float kOnePassMin = 4e-3f;   // (sigma / mu)^2 below which the two-pass form is used

// One half (64 rows) of a key's column into registers: A'[r] for rows h0..h0+63
// (rows that do not see the key -- causal -- or past n give 0).
template <bool kFull>
__device__ __forceinline__ void col_half_values(const ScoreParams& P, const ScoreCtl& ctl,
                                                const float4* nb4, uint32_t taddr, int h0, int n,
                                                int rel, float (&v)[64]) {
  const int nh = kFull ? 64 : (n - h0 < 64 ? n - h0 : 64);   // rows of this half, >= 1
  tmem_ld32(taddr + h0, v);
  if (kFull || nh > 32) {
    tmem_ld32(taddr + h0 + 32, v + 32);
  } else {
#pragma unroll
    for (int r = 32; r < 64; ++r) v[r] = 0.f;   // not loaded: rows past n
  }
  tmem_wait_ld();
  const float2 a2 = make_float2(P.alpha, P.alpha);
#pragma unroll
  for (int r = 0; r < 64; r += 4) {
    const float4 b = nb4[(h0 + r) >> 2];
    const float2 x0 = ffma2(make_float2(v[r], v[r + 1]), a2, make_float2(b.x, b.y));
    const float2 x1 = ffma2(make_float2(v[r + 2], v[r + 3]), a2, make_float2(b.z, b.w));
    if (kFull) {
      v[r] = ex2(x0.x);
      v[r + 1] = ex2(x0.y);
      v[r + 2] = ex2(x1.x);
      v[r + 3] = ex2(x1.y);
    } else {
      // rows past n are staged as -inf: 2^-inf = 0 even where their products are
      // not finite
      v[r] = ex2(fmaxf(x0.x, -INFINITY));
      v[r + 1] = ex2(fmaxf(x0.y, -INFINITY));
      v[r + 2] = ex2(fmaxf(x1.x, -INFINITY));
      v[r + 3] = ex2(fmaxf(x1.y, -INFINITY));
    }
  }
  if (rel > 0) {
#pragma unroll
    for (int r = 0; r < 64; ++r)
      if (rel > ctl.roww[h0 + r]) v[r] = 0.f;
  }
}

// bf16 bits of two floats packed in one word (round to nearest even): lo in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// Window output: the probabilities A[r][key] = A'[r] * 2^-40 of this half's 64 rows as
// bf16 into the P^T tile (K = the tile's 128 keys, N = the 128 rows), MN-major with the
// 128-byte swizzle: rows 64h.. form the atom at h * 16 KB, key k's 128-byte row of it sits
// at (k / 8) * 1024 + (k % 8) * 128, and its 16-byte chunk c (rows 8c .. 8c + 7) at
// position c ^ (k % 8).
__device__ __forceinline__ void write_pt_half(uint8_t* pt, int key, int h0, const float (&v)[64]) {
  uint8_t* row = pt + (h0 >> 6) * kHalfBytes + (key >> 3) * 1024 + (key & 7) * 128;
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const float* x = v + 8 * c;
    const uint4 w = make_uint4(pack_bf16x2(x[0] * kColUnscale, x[1] * kColUnscale),
                               pack_bf16x2(x[2] * kColUnscale, x[3] * kColUnscale),
                               pack_bf16x2(x[4] * kColUnscale, x[5] * kColUnscale),
                               pack_bf16x2(x[6] * kColUnscale, x[7] * kColUnscale));
    *reinterpret_cast<uint4*>(row + ((c ^ (key & 7)) << 4)) = w;
  }
}

// Sum and sum of squares of a half (3 fp32 operations per element with the
// exponent's argument: the FMA pipe stays below the MUFU pipe). With the window
// output (pt != null), the half's probabilities also go to the P^T tile.
template <bool kFull, bool kAttn>
__device__ __forceinline__ void colsums_half(const ScoreParams& P, const ScoreCtl& ctl,
                                             const float4* nb4, uint32_t taddr, int h0, int n,
                                             int rel, float& sum, float& sumsq, uint8_t* pt, int key) {
  float v[64];
  col_half_values<kFull>(P, ctl, nb4, taddr, h0, n, rel, v);
  if constexpr (kAttn) write_pt_half(pt, key, h0, v);
  float2 c0 = make_float2(0.f, 0.f), c1 = c0, c2 = c0, c3 = c0;
  float2 q0 = c0, q1 = c0, q2 = c0, q3 = c0;
#pragma unroll
  for (int r = 0; r < 64; r += 8) {
    const float2 p0 = make_float2(v[r], v[r + 1]), p1 = make_float2(v[r + 2], v[r + 3]);
    const float2 p2 = make_float2(v[r + 4], v[r + 5]), p3 = make_float2(v[r + 6], v[r + 7]);
    c0 = fadd2(c0, p0);
    c1 = fadd2(c1, p1);
    c2 = fadd2(c2, p2);
    c3 = fadd2(c3, p3);
    q0 = ffma2(p0, p0, q0);
    q1 = ffma2(p1, p1, q1);
    q2 = ffma2(p2, p2, q2);
    q3 = ffma2(p3, p3, q3);
  }
  const float2 cs = fadd2(fadd2(c0, c1), fadd2(c2, c3));
  const float2 qs = fadd2(fadd2(q0, q1), fadd2(q2, q3));
  sum = cs.x + cs.y;
  sumsq = qs.x + qs.y;
}

// The same half, two passes: its sum and its sum of squared deviations from its own
// mean (no cancellation; used when the one-pass form cannot be trusted).
template <bool kFull>
__device__ __forceinline__ void colstats_half(const ScoreParams& P, const ScoreCtl& ctl,
                                              const float4* nb4, uint32_t taddr, int h0, int n,
                                              int rel, float& sum, float& m2) {
  const int nh = kFull ? 64 : (n - h0 < 64 ? n - h0 : 64);
  float v[64];
  col_half_values<kFull>(P, ctl, nb4, taddr, h0, n, rel, v);
  float2 c0 = make_float2(0.f, 0.f), c1 = c0, c2 = c0, c3 = c0;
#pragma unroll
  for (int r = 0; r < 64; r += 8) {
    c0 = fadd2(c0, make_float2(v[r], v[r + 1]));
    c1 = fadd2(c1, make_float2(v[r + 2], v[r + 3]));
    c2 = fadd2(c2, make_float2(v[r + 4], v[r + 5]));
    c3 = fadd2(c3, make_float2(v[r + 6], v[r + 7]));
  }
  const float2 cs = fadd2(fadd2(c0, c1), fadd2(c2, c3));
  sum = cs.x + cs.y;
  const float mh = sum / static_cast<float>(nh);
  float q = 0.f;
#pragma unroll
  for (int r = 0; r < 64; ++r) {
    // rows past n: no term (ctl.rowm is 1 for rows r < n, else 0)
    const float d = kFull ? v[r] - mh : (v[r] - mh) * ctl.rowm[h0 + r];
    q = fmaf(d, d, q);
  }
  m2 = q;
}

// With the window output (kAttn), every tile's probabilities go to the P^T tile in the
// tile's K stage (kbuf + stage * 32 KB; the score MMA has finished with its K), announced
// on p_full[stage]; at the end of the item group 0 reads the item's O^T accumulator
// (lane = d, column = row) into o_part[item][row][d] and hands it back on o_empty. oi
// counts the column items before this one.
template <bool kFull, bool kAttn>
__device__ __forceinline__ bool colstats_item(const ScoreParams& P, ScoreCtl& ctl,
                                              const ItemDesc& d, uint32_t slot, uint32_t& ai,
                                              uint8_t* kbuf, uint32_t& oi) {
  constexpr int kAccBufs = Cfg<kAttn>::kAccBufs;
  constexpr int kKStages = Cfg<kAttn>::kKStages;
  const int quad = (threadIdx.x >> 5) & 3;
  const int lane = threadIdx.x & 31;
  const int grp = (threadIdx.x - kEpiWarp0 * 32) >> 7;
  const int tl = quad * 32 + lane;         // key within the tile
  const int n = kFull ? kMaxRows : P.g.n_rows;
  const int W = P.g.window;
  const int tile0 = d.tile0, ntiles = d.ntiles;
  const float fn = static_cast<float>(n);
  const float inv_n = 1.0f / fn;
  const float inv_n1 = n > 1 ? 1.0f / static_cast<float>(n - 1) : 0.f;
  const float4* nb4 = reinterpret_cast<const float4*>(ctl.nbeta[slot]);
  for (int t = 0; t < ntiles; ++t, ++ai) {
    if (static_cast<int>(ai & 1u) != grp) continue;
    const uint32_t ab = ai % kAccBufs;
    if (!warp_wait(&ctl.acc_full[ab], (ai / kAccBufs) & 1u, P.wait_limit_ns, &ctl.abort))
      return false;
    tc_fence_after();
    const uint32_t taddr = ctl.tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + ab * 128u;
    const int key = (tile0 + t) * kTileKeys + tl;
    const int rel = key - (d.L - W);          // > 0: the key is inside the window
    // the column's rows in two halves of 64 (registers): one pass of sums and sums
    // of squares, m2 = sum A'^2 - (sum A')^2 / n
    const bool two = kFull || n > 64;
    float S1 = 0.f, SS = 0.f;
    uint8_t* pt = kAttn ? kbuf + (ai % kKStages) * kTileBytes : nullptr;
#pragma unroll 1
    for (int h = 0; h < (two ? 2 : 1); ++h) {
      float sh, qh;
      colsums_half<kFull, kAttn>(P, ctl, nb4, taddr, 64 * h, n, rel, sh, qh, pt, tl);
      S1 += sh;
      SS += qh;
    }
    if constexpr (kAttn) {
      if (!two) {
        // rows 64..127 are past n: their probabilities are 0
#pragma unroll
        for (int c = 0; c < 8; ++c)
          *reinterpret_cast<uint4*>(pt + kHalfBytes + (tl >> 3) * 1024 + (tl & 7) * 128 + (c << 4)) =
              make_uint4(0, 0, 0, 0);
      }
      // P^T is read by the tensor cores (async proxy) once every warp has announced it
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.p_full[ai % kKStages]);
    }
    float m2 = fmaf(-S1, S1 * inv_n, SS);
    // The one-pass form loses about (sum A'^2) * 2^-19 to rounding. It is kept while
    // sigma^2 >= kOnePassMin * mu^2, where that loss stays below 2e-4 of sigma^2;
    // otherwise (columns of nearly equal A, e.g. uniform attention) the warp takes
    // the two-pass form over the same TMEM columns, halves combined by the pairwise
    // update of the mean and the sum of squared deviations (Chan, Golub, LeVeque).
    const bool exact = !(m2 * fn * fn >= kOnePassMin * (fn - 1.f) * S1 * S1);   // NaN-safe
    if (__any_sync(0xffffffffu, exact)) {
      float hs[2] = {0.f, 0.f}, hm2[2] = {0.f, 0.f};
#pragma unroll 1
      for (int h = 0; h < (two ? 2 : 1); ++h) {
        float sh, mh2;
        colstats_half<kFull>(P, ctl, nb4, taddr, 64 * h, n, rel, sh, mh2);
        if (h == 0) { hs[0] = sh; hm2[0] = mh2; } else { hs[1] = sh; hm2[1] = mh2; }
      }
      const float n1 = kFull ? 64.f : static_cast<float>(n < 64 ? n : 64);
      const float n2 = fn - n1;
      float m2x = hm2[0] + hm2[1];
      if (two) {
        const float dd = hs[1] / n2 - hs[0] / n1;
        m2x = fmaf(dd * dd, n1 * n2 * inv_n, m2x);
      }
      if (exact) m2 = m2x;
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl.acc_empty[ab]);
    const float mu = S1 * inv_n * kColUnscale;
    const float sigma = sqrtf(fmaxf(m2, 0.f) * inv_n1) * kColUnscale;
    if (key < d.L) {
      __stcs(&P.mu[d.mu_off + key], mu);
      __stcs(&P.sigma[d.mu_off + key], sigma);
    }
  }
  if constexpr (kAttn) {
    if (grp == 0) {
      // the item's O^T (lane = d, column = row) into o_part[item][row][d]
      if (!warp_wait(&ctl.o_full, oi & 1u, P.wait_limit_ns, &ctl.abort)) return false;
      tc_fence_after();
      const uint32_t taddr = ctl.tmem_base + (static_cast<uint32_t>(quad * 32) << 16) + kOCol;
      float* dst = P.o_part + d.p * (kMaxRows * kHeadDim) + tl;
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(taddr + 32u * c, v);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) __stcg(dst + (32 * c + j) * kHeadDim, v[j]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.o_empty);
    }
    ++oi;
  }
  return true;
}

// ---------------------------------------------------------------- sync warp

// One round of loads of a unit's tagged normalisers (4 rows per lane; relaxed GPU-scope
// loads, so that every poll reads memory again); rows past n read as ready.
__device__ __forceinline__ void load_beta(const ScoreParams& P, int64_t unit, unsigned long long w[4]) {
  const int r0 = 4 * (threadIdx.x & 31);
#pragma unroll
  for (int k = 0; k < 4; ++k)
    w[k] = (r0 + k < P.g.n_rows) ? ld_relaxed_gpu_u64(&P.beta[unit * kMaxRows + r0 + k]) : (1ull << 32);
}

// If every row of w is tagged ready, stage -beta for the epilogue and return true.
__device__ __forceinline__ bool stage_beta(const ScoreParams& P, ScoreCtl& ctl,
                                           const unsigned long long w[4], uint32_t slot) {
  const int lane = threadIdx.x & 31;
  const int n = P.g.n_rows;
  const int r0 = 4 * lane;
  bool ready = true;
#pragma unroll
  for (int k = 0; k < 4; ++k) ready = ready && (w[k] >> 32) != 0ull;
  if (!__all_sync(0xffffffffu, ready)) return false;
  float4 b;
  b.x = r0 + 0 < n ? kColScale - __uint_as_float(static_cast<uint32_t>(w[0])) : -INFINITY;
  b.y = r0 + 1 < n ? kColScale - __uint_as_float(static_cast<uint32_t>(w[1])) : -INFINITY;
  b.z = r0 + 2 < n ? kColScale - __uint_as_float(static_cast<uint32_t>(w[2])) : -INFINITY;
  b.w = r0 + 3 < n ? kColScale - __uint_as_float(static_cast<uint32_t>(w[3])) : -INFINITY;
  reinterpret_cast<float4*>(ctl.nbeta[slot])[lane] = b;
  return true;
}

// Phase-0 item: merge the two groups' (m, Z) per row, publish them and count the
// item. Returns whether it was the unit's last item to arrive. When the next ring
// item is a phase-1 item not yet staged (next_unit >= 0), its normalisers are loaded
// before the publication's fence and checked after its atomic (the round trips
// overlap); *next_staged tells whether they were ready and are now staged.
__device__ __forceinline__ bool sync_rowstats(const ScoreParams& P, ScoreCtl& ctl,
                                              const ItemDesc& d, uint32_t slot, int64_t next_unit,
                                              uint32_t next_slot, bool* next_staged) {
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
  unsigned long long w[4];
  if (next_unit >= 0) load_beta(P, next_unit, w);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = lane + 32 * k;
    if (row < n) P.partial[d.p * kMaxRows + row] = mz[k];
  }
  __threadfence();
  __syncwarp();
  int last = 0;
  if (lane == 0 && !(P.fault == 1 && d.unit == 0)) {
    const uint32_t old = atomicAdd(&P.counts[d.unit], 1u);
    last = (old == static_cast<uint32_t>(d.splits - 1));
  }
  *next_staged = next_unit >= 0 && stage_beta(P, ctl, w, next_slot);
  return __shfl_sync(0xffffffffu, last, 0) != 0;
}

// Merge warp: fold all of a unit's (m, Z) partials into beta_r = m + log2 Z and
// publish each row's beta with its ready tag. The partials of a unit are contiguous
// (1 KB per item) and come in by bulk copies of up to kMergeBatch items.
template <bool kAttn>
__device__ __forceinline__ bool merge_unit(const ScoreParams& P, ScoreCtl& ctl, const MergeJob& u,
                                           float2 (*mbuf)[kMaxRows], uint32_t& phase) {
  constexpr int kMergeBatch = Cfg<kAttn>::kMergeBatch;
  const int lane = threadIdx.x & 31;
  const int n = P.g.n_rows;
  __threadfence();
  float M[4], Z[4];   // running (max, sum) per row, log2 units
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    M[k] = -INFINITY;
    Z[k] = 0.f;
  }
  for (int s0 = 0; s0 < u.splits; s0 += kMergeBatch) {
    const int cnt = u.splits - s0 < kMergeBatch ? u.splits - s0 : kMergeBatch;
    if (lane == 0) {
      // the other CTAs' partials (acquired above) and this warp's reads of the
      // previous batch come before the copy
      fence_proxy_async();
      const uint32_t bytes = static_cast<uint32_t>(cnt) * kMaxRows * sizeof(float2);
      mbar_arrive_expect_tx(&ctl.merge_bar, bytes);
      bulk_load(&mbuf[0][0], &P.partial[(u.item0 + s0) * kMaxRows], bytes, &ctl.merge_bar);
    }
    if (!warp_wait(&ctl.merge_bar, phase, P.wait_limit_ns, &ctl.abort)) return false;
    phase ^= 1u;
    // all loads first (unconditional, masked afterwards), then the max, then every
    // partial rescaled to it: the loads and the exponentials are independent
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int row = lane + 32 * k;
      float2 e[kMergeBatch];
#pragma unroll
      for (int j = 0; j < kMergeBatch; ++j) {
        const float2 x = mbuf[j][row];
        e[j] = j < cnt ? x : make_float2(-INFINITY, 0.f);
      }
      float mb = M[k];
#pragma unroll
      for (int j = 0; j < kMergeBatch; ++j) mb = fmaxf(mb, e[j].x);
      if (row >= n || mb == -INFINITY) continue;
      float z0 = M[k] == -INFINITY ? 0.f : Z[k] * ex2(M[k] - mb), z1 = 0.f, z2 = 0.f, z3 = 0.f;
#pragma unroll
      for (int j = 0; j < kMergeBatch; j += 4) {
        z0 = fmaf(e[j].y, ex2(e[j].x - mb), z0);   // ex2(-inf) = 0 for empty partials
        if (j + 1 < kMergeBatch) z1 = fmaf(e[j + 1].y, ex2(e[j + 1].x - mb), z1);
        if (j + 2 < kMergeBatch) z2 = fmaf(e[j + 2].y, ex2(e[j + 2].x - mb), z2);
        if (j + 3 < kMergeBatch) z3 = fmaf(e[j + 3].y, ex2(e[j + 3].x - mb), z3);
      }
      M[k] = mb;
      Z[k] = (z0 + z1) + (z2 + z3);
    }
    __syncwarp();
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int row = lane + 32 * k;
    if (row < n) {
      // one 64-bit store: a reader sees either the cleared word or (beta, 1)
      const float b = M[k] + lg2(Z[k]);
      const unsigned long long word =
          (1ull << 32) | static_cast<unsigned long long>(__float_as_uint(b));
      __stcg(&P.beta[u.unit * kMaxRows + row], word);
    }
  }
  return true;
}

// Phase-1 item: one round of loads of the unit's normalisers. Each row's word carries
// its own ready tag; when every row is ready, -beta is staged in shared memory for
// the epilogue and true is returned.
__device__ __forceinline__ bool try_stage_beta(const ScoreParams& P, ScoreCtl& ctl, int64_t unit,
                                               uint32_t slot) {
  unsigned long long w[4];
  load_beta(P, unit, w);
  return stage_beta(P, ctl, w, slot);
}

// Phase-1 item with given normalisers (P.lse, natural log): stage -beta = -log2(e) * lse
// of the unit's rows; nothing to wait for.
__device__ __forceinline__ void stage_lse(const ScoreParams& P, ScoreCtl& ctl, int64_t unit, uint32_t slot) {
  constexpr float kLog2e = 1.4426950408889634f;
  const UnitInfo u = unit_info(P.g, unit);
  const float* l = P.lse + u.q_row0;
  const int n = P.g.n_rows;
  const int r0 = 4 * (threadIdx.x & 31);
  float4 b;
  b.x = r0 + 0 < n ? fmaf(-kLog2e, l[r0 + 0], kColScale) : -INFINITY;
  b.y = r0 + 1 < n ? fmaf(-kLog2e, l[r0 + 1], kColScale) : -INFINITY;
  b.z = r0 + 2 < n ? fmaf(-kLog2e, l[r0 + 2], kColScale) : -INFINITY;
  b.w = r0 + 3 < n ? fmaf(-kLog2e, l[r0 + 3], kColScale) : -INFINITY;
  reinterpret_cast<float4*>(ctl.nbeta[slot])[threadIdx.x & 31] = b;
}

// Phase-1 item: wait (bounded) for the unit's merged statistics and stage -beta.
__device__ __forceinline__ bool sync_colstats(const ScoreParams& P, ScoreCtl& ctl, int64_t unit,
                                              uint32_t slot) {
  const int lane = threadIdx.x & 31;
  uint64_t t0 = 0;   // timer read on the first miss only
  const volatile uint32_t* errw = P.err;
  uint32_t ns = 32;
  for (;;) {
    if (try_stage_beta(P, ctl, unit, slot)) return true;
    int give_up = 0;
    if (lane == 0) {
      const uint64_t now = global_timer_ns();
      if (t0 == 0) t0 = now;
      give_up = (*errw != 0u || ctl.abort || now - t0 > P.wait_limit_ns) ? 1 : 0;
    }
    if (__shfl_sync(0xffffffffu, give_up, 0)) return false;
    __nanosleep(ns);
    if (ns < 512) ns *= 2;
  }
}

// ---------------------------------------------------------------- kernel

// kAttn: the window output variant (tm_v maps v; for the plain kernel tm_v is unused).
template <bool kFull, bool kAttn>
__global__ void __launch_bounds__(kThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ ScoreParams P) {
  constexpr int kQBufs = Cfg<kAttn>::kQBufs;
  constexpr int kKStages = Cfg<kAttn>::kKStages;
  constexpr int kAccBufs = Cfg<kAttn>::kAccBufs;
  __shared__ ScoreCtl ctl;
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* qbuf = tiles;                             // kQBufs x 32 KB
  uint8_t* kbuf = tiles + kQBufs * kTileBytes;       // kKStages x 32 KB
  uint8_t* vbuf = kbuf + kKStages * kTileBytes;      // kVStages x 32 KB (window output)
  // partials being merged (bulk-copy destination, 1 KB aligned)
  float2 (*mbuf)[kMaxRows] =
      reinterpret_cast<float2 (*)[kMaxRows]>(vbuf + Cfg<kAttn>::kVStages * kTileBytes);

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
    for (int i = 0; i < kMergeSlots; ++i) {
      mbar_init(&ctl.merge_full[i], 1);
      mbar_init(&ctl.merge_empty[i], 1);
    }
    if constexpr (kAttn) {
      for (int i = 0; i < Cfg<kAttn>::kVStages; ++i) {
        mbar_init(&ctl.v_full[i], 1);
        mbar_init(&ctl.v_empty[i], 1);
      }
      for (int i = 0; i < kKStages; ++i) mbar_init(&ctl.p_full[i], 4);   // the tile's 4 warps
      mbar_init(&ctl.o_full, 1);
      mbar_init(&ctl.o_empty, 4);                                          // group 0
    }
    mbar_init(&ctl.merge_bar, 1);
    ctl.abort = 0;
    fence_mbar_init();
    prefetch_tensormap(&tm_q);
    prefetch_tensormap(&tm_k);
    if (kAttn) prefetch_tensormap(&tm_v);
  }
  if (threadIdx.x < kMaxRows) {
    ctl.roww[threadIdx.x] = threadIdx.x % P.g.window;
    ctl.rowm[threadIdx.x] = static_cast<int>(threadIdx.x) < P.g.n_rows ? 1.f : 0.f;
  }
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
      uint32_t it = 0, qi = 0, ki = 0, vi = 0;
      // bit i: buffer / stage i has been loaded at least once, and the parity of its last load
      uint32_t q_used = 0, k_used = 0, q_last = 0, k_last = 0, v_used = 0, v_last = 0;
      const uint64_t pol_keep = l2_policy_evict_last();
      const uint64_t pol_drop = l2_policy_evict_first();
      bool ok = true;
      // Own items p_j = c + j*G. Sequence: phase 0 of p_j while j - jc <= lag, else
      // phase 1 of p_jc; phase 1 of p_jc therefore follows phase 0 of p_(jc+lag).
      const int64_t G = gridDim.x;
      const int64_t own = (n1 - blockIdx.x + G - 1) / G;
      int64_t jr = 0, jc = 0;
      for (;;) {
        Claim cl;
        bool have = true;
        if (ctl.abort) {
          have = false;
        } else if (!P.lse && jr < own && jr - jc <= P.lag) {
          // (with given normalisers there are no phase-0 items)
          cl.phase = 0;
          cl.p = blockIdx.x + jr * G;
          ++jr;
        } else if (jc < own) {
          cl.phase = 1;
          cl.p = blockIdx.x + jc * G;
          ++jc;
        } else {
          have = false;
        }
        const uint32_t slot = it % kItemSlots;
        if (!mbar_wait(&ctl.item_empty[slot], ((it / kItemSlots) & 1u) ^ 1u,
                       P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        ItemDesc d;
        UnitInfo u;
        if (have) {
          int split;
          u = unit_info(P.g, item_unit(P.g, cl.p, &split));
          d.p = cl.p;
          d.unit = u.unit;
          d.mu_off = u.mu_off;
          d.item0 = u.item0;
          d.phase = cl.phase;
          item_range(u, split, &d.tile0, &d.ntiles);
          d.L = u.L;
          d.splits = u.splits;
          d.tok0 = static_cast<int32_t>(u.tok0);
          d.kvh = u.kvh;
          d.layer = u.layer;
        } else {
          d.p = -1;
        }
        ctl.item_ring[slot] = d;
        mbar_arrive(&ctl.item_full[slot]);
        ++it;
        if (!have) break;
        const uint32_t qb = qi % kQBufs;
        if (!mbar_wait(&ctl.q_empty[qb], ((qi / kQBufs) & 1u) ^ 1u,
                       P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&ctl.q_full[qb], kTileBytes);
        tma_load_2d(qbuf + qb * kTileBytes, &tm_q, 0, static_cast<int32_t>(u.q_row0), &ctl.q_full[qb]);
        tma_load_2d(qbuf + qb * kTileBytes + kHalfBytes, &tm_q, 64, static_cast<int32_t>(u.q_row0),
                    &ctl.q_full[qb]);
        q_used |= 1u << qb;
        q_last = (q_last & ~(1u << qb)) | (((qi / kQBufs) & 1u) << qb);
        ++qi;
        const int tile0 = d.tile0, ntiles = d.ntiles;
        const uint64_t pol = cl.phase == 0 ? pol_keep : pol_drop;
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t ks = ki % kKStages;
          if (!mbar_wait(&ctl.k_empty[ks], ((ki / kKStages) & 1u) ^ 1u,
                         P.wait_limit_ns, &ctl.abort)) {
            ok = false;
            break;
          }
          const int32_t y = d.tok0 + (tile0 + t) * kTileKeys;
          mbar_arrive_expect_tx(&ctl.k_full[ks], kTileBytes);
          tma_load_4d_hint(kbuf + ks * kTileBytes, &tm_k, 0, y, d.kvh, d.layer, &ctl.k_full[ks], pol);
          tma_load_4d_hint(kbuf + ks * kTileBytes + kHalfBytes, &tm_k, 64, y, d.kvh, d.layer,
                           &ctl.k_full[ks], pol);
          k_used |= 1u << ks;
          k_last = (k_last & ~(1u << ks)) | (((ki / kKStages) & 1u) << ks);
          ++ki;
          if constexpr (kAttn) {
            if (cl.phase == 1) {
              // the tile's values for the window output (streamed once, from HBM)
              const uint32_t vs = vi % Cfg<kAttn>::kVStages;
              const uint32_t vpar = (vi / Cfg<kAttn>::kVStages) & 1u;
              if (!mbar_wait(&ctl.v_empty[vs], vpar ^ 1u, P.wait_limit_ns, &ctl.abort)) {
                ok = false;
                break;
              }
              mbar_arrive_expect_tx(&ctl.v_full[vs], kTileBytes);
              tma_load_4d_hint(vbuf + vs * kTileBytes, &tm_v, 0, y, d.kvh, d.layer, &ctl.v_full[vs],
                               pol_drop);
              tma_load_4d_hint(vbuf + vs * kTileBytes + kHalfBytes, &tm_v, 64, y, d.kvh, d.layer,
                               &ctl.v_full[vs], pol_drop);
              v_used |= 1u << vs;
              v_last = (v_last & ~(1u << vs)) | (vpar << vs);
              ++vi;
            }
          }
        }
        if (!ok) break;
      }
      if (!ok) set_error(P, ctl, 1u);
      // no bulk copy may still be writing shared memory when the CTA exits
      volatile int no_abort = 0;
      for (int i = 0; i < kQBufs; ++i)
        if ((q_used >> i) & 1u) mbar_wait(&ctl.q_full[i], (q_last >> i) & 1u, P.wait_limit_ns, &no_abort);
      for (int i = 0; i < kKStages; ++i)
        if ((k_used >> i) & 1u) mbar_wait(&ctl.k_full[i], (k_last >> i) & 1u, P.wait_limit_ns, &no_abort);
      for (int i = 0; i < Cfg<kAttn>::kVStages; ++i)
        if ((v_used >> i) & 1u) mbar_wait(&ctl.v_full[i], (v_last >> i) & 1u, P.wait_limit_ns, &no_abort);
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
      // window output: the O^T MMA of a column tile runs one tile behind its score MMA
      // (its P^T must be written first); pend_* describe the tile waiting for it
      const uint32_t vaddr = smem_u32(vbuf);
      uint32_t vi = 0, oi = 0, pcnt[kMaxKStages] = {}, last_opar = 0;
      int pend_ks = -1, pend_vs = 0, o_issued = 0;
      uint32_t pend_vpar = 0;
      bool pend_first = false;
      auto issue_pv = [&]() -> bool {
        if (!mbar_wait(&ctl.p_full[pend_ks], pcnt[pend_ks] & 1u, P.wait_limit_ns, &ctl.abort) ||
            !mbar_wait(&ctl.v_full[pend_vs], pend_vpar, P.wait_limit_ns, &ctl.abort) ||
            (pend_first && !mbar_wait(&ctl.o_empty, (oi & 1u) ^ 1u, P.wait_limit_ns, &ctl.abort)))
          return false;
        ++pcnt[pend_ks];
        tc_fence_after();
        const uint32_t va = vaddr + pend_vs * kTileBytes, pa = kaddr + pend_ks * kTileBytes;
#pragma unroll
        for (int j = 0; j < kHeadDim / 16; ++j)   // 16 keys per MMA: 2 KB of each operand
          tc_mma_bf16(ctl.tmem_base + kOCol, sw128_mn_desc(va + 2048u * j, kMNLbo, kMNSbo),
                      sw128_mn_desc(pa + 2048u * j, kMNLbo, kMNSbo), kIdescMN,
                      (pend_first && j == 0) ? 0u : 1u);
        tc_commit(&ctl.k_empty[pend_ks]);
        tc_commit(&ctl.v_empty[pend_vs]);
        pend_ks = -1;
        return true;
      };
      for (;;) {
        const uint32_t slot = it % kItemSlots;
        if (!mbar_wait(&ctl.item_full[slot], (it / kItemSlots) & 1u,
                       P.wait_limit_ns, &ctl.abort)) {
          ok = false;
          break;
        }
        const int phase = ctl.item_ring[slot].phase;
        const int ntiles = ctl.item_ring[slot].ntiles;
        const bool end = ctl.item_ring[slot].p < 0;
        mbar_arrive(&ctl.item_empty[slot]);
        ++it;
        if (end) break;
        const uint32_t qb = qi % kQBufs;
        if (!mbar_wait(&ctl.q_full[qb], (qi / kQBufs) & 1u, P.wait_limit_ns,
                       &ctl.abort)) {
          ok = false;
          break;
        }
        ++qi;
        for (int t = 0; t < ntiles; ++t) {
          const uint32_t ks = ki % kKStages;
          const uint32_t ab = ai % kAccBufs;
          if (!mbar_wait2(&ctl.k_full[ks], (ki / kKStages) & 1u, &ctl.acc_empty[ab],
                          ((ai / kAccBufs) & 1u) ^ 1u, P.wait_limit_ns, &ctl.abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = ctl.tmem_base + ab * 128u;
          // operand roles per phase are chosen once per tile: the issue loop below is
          // branch-free (a single thread issues, so every extra instruction costs MMA rate)
          const uint32_t qs = qaddr + qb * kTileBytes, kss = kaddr + ks * kTileBytes;
          const uint64_t ad = sw128_desc(phase == 0 ? qs : kss);
          const uint64_t bd = sw128_desc(phase == 0 ? kss : qs);
#pragma unroll
          for (int j = 0; j < kHeadDim / 16; ++j) {
            // the descriptor's start-address field counts 16-byte units
            const uint64_t off = ((j >> 2) * kHalfBytes + (j & 3) * 32u) >> 4;
            tc_mma_bf16(d_tmem, ad + off, bd + off, kIdesc, j > 0 ? 1u : 0u);
          }
          if (!kAttn || phase == 0) tc_commit(&ctl.k_empty[ks]);
          tc_commit(&ctl.acc_full[ab]);
          issued = 1;
          last_ab = ab;
          last_par = (ai / kAccBufs) & 1u;
          if constexpr (kAttn) {
            if (phase == 1) {
              if (pend_ks >= 0 && !issue_pv()) {
                ok = false;
                break;
              }
              pend_ks = static_cast<int>(ks);
              pend_vs = static_cast<int>(vi % Cfg<kAttn>::kVStages);
              pend_vpar = (vi / Cfg<kAttn>::kVStages) & 1u;
              pend_first = t == 0;
              ++vi;
            }
          }
          ++ki;
          ++ai;
        }
        if (!ok) break;
        if constexpr (kAttn) {
          if (phase == 1) {
            // the item's last O^T MMA, then O^T goes to the epilogue
            if (!issue_pv()) {
              ok = false;
              break;
            }
            tc_commit(&ctl.o_full);
            o_issued = 1;
            last_opar = oi & 1u;
            ++oi;
          }
        }
        tc_commit(&ctl.q_empty[qb]);
      }
      if (!ok) set_error(P, ctl, 1u);
      // the MMAs must have finished before TMEM is released
      volatile int no_abort = 0;
      if (issued)
        mbar_wait(&ctl.acc_full[last_ab], last_par, P.wait_limit_ns, &no_abort);
      if (kAttn && o_issued) mbar_wait(&ctl.o_full, last_opar, P.wait_limit_ns, &no_abort);
    }
  } else if (warp == kSyncWarp) {
    // ------------------------------------------------------------ sync warp
    uint32_t it = 0, mj = 0;
    // hand a unit (or -1: no more units) to the merge warp
    auto post_merge = [&](const MergeJob& job) -> bool {
      const uint32_t ms = mj % kMergeSlots;
      if (!warp_wait(&ctl.merge_empty[ms], ((mj / kMergeSlots) & 1u) ^ 1u, P.wait_limit_ns, &ctl.abort))
        return false;
      if (lane == 0) {
        ctl.merge_job[ms] = job;
        mbar_arrive(&ctl.merge_full[ms]);
      }
      ++mj;
      return true;
    };
    bool staged = false;   // item `it` is a phase-1 item already staged and released
    for (;;) {
      if (staged) {
        // its slot may already hold a later item: never wait on it again
        staged = false;
        ++it;
        continue;
      }
      const uint32_t slot = it % kItemSlots;
      const uint32_t par = (it / kItemSlots) & 1u;
      if (!warp_wait(&ctl.item_full[slot], par, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const ItemDesc d = ctl.item_ring[slot];
      if (d.p < 0) {
        MergeJob none;
        none.unit = -1;
        if (!post_merge(none)) set_error(P, ctl, 1u);
        break;
      }
      bool ok = true;
      bool next_staged = false;
      if (d.phase == 0) {
        if (lane == 0) mbar_arrive(&ctl.beta_full[slot]);      // nothing to stage
        // While the epilogue finishes this item, stage the next item's normalisers
        // if it is a phase-1 item whose unit is already merged.
        const uint32_t nslot = (it + 1) % kItemSlots;
        const uint32_t npar = ((it + 1) / kItemSlots) & 1u;
        bool next_checked = false;
        int64_t next_unit = -1;   // the next item is a phase-1 item of this unit, not staged
        uint64_t t0 = 0;
        for (;;) {
          // test_wait, not try_wait: the loop also polls the next item's normalisers and
          // must not be suspended while the epilogue finishes
          if (__all_sync(0xffffffffu, mbar_test_wait(&ctl.pub_full[slot], par))) break;
          if (!next_checked && __all_sync(0xffffffffu, mbar_test_wait(&ctl.item_full[nslot], npar))) {
            const int64_t pn = ctl.item_ring[nslot].p;
            const int phn = ctl.item_ring[nslot].phase;
            if (pn < 0 || phn == 0) {
              next_checked = true;
            } else {
              next_unit = ctl.item_ring[nslot].unit;
              if (try_stage_beta(P, ctl, next_unit, nslot)) {
                next_unit = -1;
                // the sync warp's whole part in that item is done: release it now
                next_checked = next_staged = true;
                __syncwarp();
                if (lane == 0) {
                  mbar_arrive(&ctl.beta_full[nslot]);
                  mbar_arrive(&ctl.item_empty[nslot]);
                }
              }
            }
          }
          int give_up = 0;
          if (lane == 0) {
            const uint64_t now = global_timer_ns();
            if (t0 == 0) t0 = now;
            give_up = (ctl.abort || now - t0 > P.wait_limit_ns) ? 1 : 0;
          }
          if (__shfl_sync(0xffffffffu, give_up, 0)) {
            ok = false;
            break;
          }
        }
        bool late_staged = false;
        const bool last = ok && sync_rowstats(P, ctl, d, slot, next_checked ? -1 : next_unit, nslot,
                                              &late_staged);
        if (late_staged) {
          // staged after the publication: release that item now as well
          next_staged = true;
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&ctl.beta_full[nslot]);
            mbar_arrive(&ctl.item_empty[nslot]);
          }
        }
        if (last) {                                              // the slot was handed back early
          MergeJob job;
          job.unit = d.unit;
          job.item0 = d.item0;
          job.splits = d.splits;
          job.pad = 0;
          ok = post_merge(job);
        }
      } else {
        if (P.lse)
          stage_lse(P, ctl, d.unit, slot);
        else
          ok = sync_colstats(P, ctl, d.unit, slot);
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
      staged = next_staged;
      ++it;
    }
  } else if (warp == kMergeWarp) {
    // ------------------------------------------------------------ merge warp
    uint32_t mj = 0, mphase = 0;
    for (;;) {
      const uint32_t ms = mj % kMergeSlots;
      if (!warp_wait(&ctl.merge_full[ms], (mj / kMergeSlots) & 1u, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const MergeJob job = ctl.merge_job[ms];
      if (job.unit < 0) break;
      if (!merge_unit<kAttn>(P, ctl, job, mbuf, mphase)) {
        set_error(P, ctl, 1u);
        // no bulk copy may still be writing shared memory when the CTA exits
        volatile int no_abort = 0;
        if (lane == 0) mbar_wait(&ctl.merge_bar, mphase, P.wait_limit_ns, &no_abort);
        break;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl.merge_empty[ms]);
      ++mj;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    uint32_t it = 0, ai = 0, oi = 0;
    for (;;) {
      const uint32_t slot = it % kItemSlots;
      const uint32_t par = (it / kItemSlots) & 1u;
      if (!warp_wait(&ctl.item_full[slot], par, P.wait_limit_ns, &ctl.abort)) {
        set_error(P, ctl, 1u);
        break;
      }
      const ItemDesc d = ctl.item_ring[slot];
      if (d.p < 0) break;
      bool ok;
      if (d.phase == 0) {
        ok = rowstats_item<kFull, kAttn>(P, ctl, d, slot, ai);
      } else {
        ok = warp_wait(&ctl.beta_full[slot], par, P.wait_limit_ns, &ctl.abort) &&
             colstats_item<kFull, kAttn>(P, ctl, d, slot, ai, kbuf, oi);
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


// Window output, last step: O of unit u's window rows = the sum of its column items'
// partials (fp32), written as bf16 in q_win's layout (row r of the unit at q_row0 + r).
__global__ void __launch_bounds__(kHeadDim) attn_finish_kernel(const __grid_constant__ Geometry g,
                                                               const float* o_part, uint16_t* o_win) {
  wait_previous_kernel();   // the partials come from the score kernel launched before
  const UnitInfo u = unit_info(g, blockIdx.x);
  const int j = threadIdx.x;   // head dimension
  for (int r = 0; r < g.n_rows; ++r) {
    float acc = 0.f;
    for (int s = 0; s < u.splits; ++s)
      acc += __ldcs(o_part + ((u.item0 + s) * kMaxRows + r) * kHeadDim + j);
    uint32_t w;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w) : "f"(0.f), "f"(acc));
    o_win[(u.q_row0 + r) * kHeadDim + j] = static_cast<uint16_t>(w & 0xFFFFu);
  }
}

template <bool kAttn>
cudaError_t launch_score_variant(bool full, const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                                 const CUtensorMap& tm_v, const ScoreParams& p, int ctas, cudaStream_t stream) {
  auto* fn = full ? score_kernel<true, kAttn> : score_kernel<false, kAttn>;
  constexpr size_t smem = Cfg<kAttn>::kDynSmem;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  // CTAs wait on each other's row statistics: all of them must be resident at once
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fn, tm_q, tm_k, tm_v, p);
}

}  // namespace

cudaError_t launch_score(const kve_plan& plan, const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                         const CUtensorMap* tm_v, const ScoreParams& p, int ctas, cudaStream_t stream) {
  const bool full = plan.geo.n_rows == kMaxRows;
  if (!tm_v) return launch_score_variant<false>(full, tm_q, tm_k, tm_k, p, ctas, stream);
  return launch_score_variant<true>(full, tm_q, tm_k, *tm_v, p, ctas, stream);
}

cudaError_t launch_attn_finish(const kve_plan& plan, const float* o_part, uint16_t* o_win,
                               cudaStream_t stream) {
  return launch_after_previous(attn_finish_kernel, dim3(static_cast<unsigned>(plan.geo.n_units)),
                               dim3(kHeadDim), 0, stream, plan.geo, o_part, o_win);
}

}  // namespace kve
