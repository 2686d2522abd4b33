// Selector kernel: step 3 of the eviction step, one CTA per unit.
//
//  1. max-pool mu and sigma over the candidate tokens 0 .. Lc-1 (Section 3.1 keeps
//     the baselines' pooling; odd kernel, stride 1, window clipped to the range)
//     and form the base score s_i = mu_i + lambda1 sigma_i (Eq. 2 without corr);
//     s is stored as an order-preserving 32-bit key in the workspace;
//  2. find the C = min(factor*B, Lc) largest keys (Section 3.2: the greedy runs on
//     the top 4B tokens) by an MSB-first radix select with 12/12/8-bit digits;
//     ties at the cut go to the lower positions;
//  3. normalise s~ = s / max(max s, eps) (Eq. 5) and stage the candidate keys
//     (bf16) and their inverse norms in shared memory;
//  4. admit min(B, C) candidates greedily (Eq. 5): value s~ + lambda2 corr, ties to
//     the lower position (the argmax compares position << 9 | slot after the value);
//     after every admission j, corr_i <- max(corr_i, cos(k_i, k_j)), which is Eq. 4
//     for the grown set (corr starts at 0, which is both corr(i, {}) and the clamp
//     at 0);
//  5. write the admitted positions ascending (and optionally in admission order,
//     with the best-minus-second margin of every admission).
// The block has one thread per pool slot (256 for C <= 256, else 512). A launch for
// several coefficient profiles (Section 3.3 re-selects for every profile a search
// tries; mu and sigma do not depend on them) runs one CTA per (unit, profile), the
// profile's coefficients and scratch taken from a table in the kernel parameters.
#include <mutex>

#include "kve_internal.h"
#include "kve_ptx.cuh"

namespace kve {
namespace {

constexpr int kChunks = kHeadDim / 8;   // 16-byte chunks of a key row
constexpr int kRowChunks = kChunks + 1; // staged row pitch (272 bytes): the 8 rows of an
                                        // mma fragment load fall on distinct banks
constexpr int kRowWords = 4 * kRowChunks;
constexpr int kBins = 4096;             // radix digits of the first two passes
constexpr int kPoolRun = 7;             // consecutive pooled outputs per run (odd: the
                                        // runs of a warp start on distinct banks)
constexpr int kPoolRuns = 2;            // runs per thread and tile
constexpr int kBatch = 16;              // key loads in flight per thread
constexpr int kTieCap = 2048;           // cut ties gathered in shared memory

__device__ __forceinline__ uint32_t ord_key(float f) {
  const uint32_t u = __float_as_uint(f + 0.0f);   // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// max of three floats in one instruction
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// 1/sqrt(x) for x > 0: the hardware estimate refined by one Newton-Raphson step,
// y <- y + y (1 - x y^2) / 2 (within about an ulp); x below 2^-64 is scaled by 2^64
// first, so that the estimate never sees a subnormal argument.
__device__ __forceinline__ float inv_sqrt(float x) {
  const bool tiny = x < 0x1p-64f;
  const float xs = tiny ? x * 0x1p64f : x;
  const float y = rsqrtf(xs);
  const float e = fmaf(-xs * y, y, 1.0f);
  const float r = fmaf(0.5f * y, e, y);
  return tiny ? r * 0x1p32f : r;
}

__device__ __forceinline__ float unord_key(uint32_t k) {
  const uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  return __uint_as_float(u);
}

template <int NT>
struct SelSmall {
  uint32_t warp_tot[NT / 32];
  uint32_t red[2][NT / 32][4];   // per warp: best key, best slot, second key
  uint32_t prefix, need, cnt, maxkey, teq, ncand;
};

// (key, position) pairs of the threshold bin staged in shared memory, after the
// finer-digit histogram in the `big` region
template <int NT>
__host__ __device__ constexpr uint32_t kCandCap() {
  return static_cast<uint32_t>((kRowChunks * NT * sizeof(uint4) - kBins * sizeof(uint32_t)) /
                               (sizeof(uint32_t) + sizeof(int32_t)));
}

// Exclusive prefix count of `flag` over the block in thread order; the block
// total is returned in *total (all threads).
template <int NT>
__device__ __forceinline__ uint32_t block_excl_count(bool flag, SelSmall<NT>& sh, uint32_t* total) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bal = __ballot_sync(0xffffffffu, flag);
  const uint32_t in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) sh.warp_tot[warp] = __popc(bal);
  __syncthreads();
  uint32_t before = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) {
    const uint32_t x = sh.warp_tot[w];
    if (w < warp) before += x;
    tot += x;
  }
  __syncthreads();
  *total = tot;
  return before + in_warp;
}

// Exclusive suffix sum of `x` over the block (sum over higher thread indices).
template <int NT>
__device__ __forceinline__ uint32_t block_excl_suffix(uint32_t x, SelSmall<NT>& sh) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_down_sync(0xffffffffu, incl, o);
    if (lane + o < 32) incl += y;
  }
  if (lane == 0) sh.warp_tot[warp] = incl;   // warp total
  __syncthreads();
  uint32_t after = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w)
    if (w > warp) after += sh.warp_tot[w];
  __syncthreads();
  return incl - x + after;
}

// Step 4 in the selection's CTA (P.k_out set): unit u's compact cache [B + W][d] as the
// gather kernel writes it. Rows r < nvalid are the kept candidates in ascending position
// (rpos[r]; their key rows are still staged in shared memory, row rslot[r]); rows
// m .. m+W-1 are the window tokens Lc .. L-1; every other row is zero. A half-warp
// copies a 256-byte row with 16-byte accesses; all loads of a batch are in flight before
// its first store. The copy is bit-exact.
template <int NT>
__device__ __forceinline__ void write_compact_cache(const SelectParams& P, const UnitInfo& u, int Lc, int m,
                                                    int nvalid, const int32_t* rpos, const int32_t* rslot,
                                                    const uint4* krow) {
  constexpr int kRowsPerPass = NT / 16;
  constexpr int kPasses = 8;
  const int W = P.g.window;
  const int rows = P.budget + W;
  const int half = threadIdx.x >> 4, lane16 = threadIdx.x & 15;
  const uint16_t* ksrc = P.k + u.k_off;
  const uint16_t* vsrc = P.v + u.v_off;
  uint4* kdst = reinterpret_cast<uint4*>(P.k_out + static_cast<int64_t>(u.unit) * rows * kHeadDim);
  uint4* vdst = reinterpret_cast<uint4*>(P.v_out + static_cast<int64_t>(u.unit) * rows * kHeadDim);
  for (int r0 = 0; r0 < rows; r0 += kPasses * kRowsPerPass) {
    uint4 kv[kPasses], vv[kPasses];
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
      const int r = r0 + p * kRowsPerPass + half;
      kv[p] = make_uint4(0, 0, 0, 0);
      vv[p] = make_uint4(0, 0, 0, 0);
      if (r < nvalid) {
        const int s = rpos[r];
        if (s >= 0 && s < Lc) {                      // never read outside the unit
          kv[p] = krow[rslot[r] * kRowChunks + lane16];
          vv[p] = __ldcs(reinterpret_cast<const uint4*>(vsrc + s * P.g.v_st) + lane16);
        }
      } else if (r >= m && r < m + W) {
        const int s = Lc + (r - m);
        kv[p] = __ldcs(reinterpret_cast<const uint4*>(ksrc + s * P.g.k_st) + lane16);
        vv[p] = __ldcs(reinterpret_cast<const uint4*>(vsrc + s * P.g.v_st) + lane16);
      }
    }
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
      const int r = r0 + p * kRowsPerPass + half;
      if (r < rows) {
        kdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = kv[p];
        vdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = vv[p];
      }
    }
  }
}

// The coefficients of one selection: those of SelectParams (kMulti = false), or
// profile first + blockIdx.y of a table (kMulti = true).
struct OneProfile {
  static constexpr bool kMulti = false;
};

template <int NT, class Prof>
__global__ void __launch_bounds__(NT, NT <= 256 ? 2 : 1) select_kernel(const __grid_constant__ SelectParams P,
                                                    const __grid_constant__ Prof prof) {
  __shared__ SelSmall<NT> sh;
  extern __shared__ __align__(16) uint8_t dyn[];
  wait_previous_kernel();   // mu and sigma come from the score kernel launched before
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  const UnitInfo u = unit_info(P.g, blockIdx.x);
  const int W = P.g.window;
  const int Lc = u.L - W;
  const int B = P.budget;                     // row stride of the outputs
  const int Bl = P.layer_budget[u.layer];     // this layer's budget, <= B
  const int C = P.cand_factor == 0 ? Lc : min(P.cand_factor * Bl, Lc);
  const int nsel = min(Bl, C);
  float lambda1 = P.lambda1[u.layer];
  float lambda2 = P.lambda2[u.layer];
  int64_t keys_off = 0, out_off = 0;   // this profile's scratch and output blocks
  if constexpr (Prof::kMulti) {
    const int row = 2 * static_cast<int>(blockIdx.y) * P.g.num_layers + u.layer;
    lambda1 = prof.lam[row];
    lambda2 = prof.lam[row + P.g.num_layers];
    keys_off = static_cast<int64_t>(prof.first + blockIdx.y) * prof.keys_stride;
    out_off = static_cast<int64_t>(prof.first + blockIdx.y) * prof.out_stride;
  }
  const float* mu = P.mu + u.mu_off;
  const float* sg = P.sigma + u.mu_off;
  uint32_t* keys = P.keys + keys_off + u.mu_off;
  const int h = P.pool_kernel / 2;

  // shared memory: [ big | cpos | ckey | spos | skey | inv | hist0 ]; `big` holds in
  // turn the pooling tiles, the radix histogram and tie list, the threshold bin's
  // (key, position) pairs, and the staged candidate keys
  uint8_t* big = dyn;
  uint4* krow = reinterpret_cast<uint4*>(big);                                  // [NT][kRowChunks]
  uint32_t* hist12 = reinterpret_cast<uint32_t*>(big);                          // [kBins] later passes
  float* tmu = reinterpret_cast<float*>(big);                                   // pooling tiles
  int32_t* cpos = reinterpret_cast<int32_t*>(big + kRowChunks * NT * sizeof(uint4));   // pool positions
  uint32_t* ckey = reinterpret_cast<uint32_t*>(cpos + NT);                      // and their keys
  int32_t* spos = reinterpret_cast<int32_t*>(ckey + NT);                        // sorted pool (or the
  uint32_t* skey = reinterpret_cast<uint32_t*>(spos + NT);                      // admitted positions)
  float* inv = reinterpret_cast<float*>(skey + NT);
  uint32_t* hist0 = reinterpret_cast<uint32_t*>(inv + NT);                      // [kBins] first pass

  for (int b = tid; b < kBins; b += NT) hist0[b] = 0;
  __syncthreads();
  // 1. pooled base score as ordered keys (and the histogram of their top 12 bits)
  // L2 policies of the pooling: the keys are read back by the scan below (evict last),
  // mu and sigma are read once here (evict first)
  const uint64_t kpol = l2_policy_evict_last();
  const uint64_t fpol = l2_policy_evict_first();
  if (h == 3) {
    // kernel 7 (the default): groups of 4 consecutive outputs that are 16-byte
    // aligned in mu, sigma and keys, each from three 16-byte loads per array (inputs
    // i-4 .. i+7); groups at the ends of the range take their inputs one by one
    const int lead = static_cast<int>(u.mu_off & 3);   // unit elements before its first aligned group
    const int ngroups = (lead + Lc + 3) / 4;
    // inputs of group q: positions 4q-lead-4 .. 4q-lead+7
    auto load_group = [&](int q, float (&xm)[12], float (&xs)[12]) {
      const int i = 4 * q - lead;
      if (i >= 4 && i + 8 <= Lc) {
        const float4* m4 = reinterpret_cast<const float4*>(mu + i - 4);
        const float4* s4 = reinterpret_cast<const float4*>(sg + i - 4);
#pragma unroll
        for (int c = 0; c < 3; ++c) {
          float4 am, as;
          asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                       : "=f"(am.x), "=f"(am.y), "=f"(am.z), "=f"(am.w) : "l"(m4 + c), "l"(fpol));
          asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                       : "=f"(as.x), "=f"(as.y), "=f"(as.z), "=f"(as.w) : "l"(s4 + c), "l"(fpol));
          xm[4 * c] = am.x;
          xm[4 * c + 1] = am.y;
          xm[4 * c + 2] = am.z;
          xm[4 * c + 3] = am.w;
          xs[4 * c] = as.x;
          xs[4 * c + 1] = as.y;
          xs[4 * c + 2] = as.z;
          xs[4 * c + 3] = as.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 12; ++j) {
          const int pj = i - 4 + j;
          const bool in = pj >= 0 && pj < Lc;          // the window is clipped to [0, Lc)
          xm[j] = in ? __ldg(mu + pj) : -INFINITY;
          xs[j] = in ? __ldg(sg + pj) : -INFINITY;
        }
      }
    };
    // output r (position i + r) pools positions i+r-3 .. i+r+3 = x[r+1 .. r+7]
    auto emit_group = [&](int q, const float (&xm)[12], const float (&xs)[12]) {
      const int i = 4 * q - lead;
      const float cm = fmaxf(max3(xm[4], xm[5], xm[6]), xm[7]);
      const float cs = fmaxf(max3(xs[4], xs[5], xs[6]), xs[7]);
      float om[4], os[4];
      om[0] = fmaxf(max3(cm, xm[1], xm[2]), xm[3]);
      om[1] = fmaxf(max3(cm, xm[2], xm[3]), xm[8]);
      om[2] = fmaxf(max3(cm, xm[3], xm[8]), xm[9]);
      om[3] = fmaxf(max3(cm, xm[8], xm[9]), xm[10]);
      os[0] = fmaxf(max3(cs, xs[1], xs[2]), xs[3]);
      os[1] = fmaxf(max3(cs, xs[2], xs[3]), xs[8]);
      os[2] = fmaxf(max3(cs, xs[3], xs[8]), xs[9]);
      os[3] = fmaxf(max3(cs, xs[8], xs[9]), xs[10]);
      uint32_t kk[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) kk[r] = ord_key(fmaf(lambda1, os[r], om[r]));
      if (i >= 0 && i + 4 <= Lc) {
        asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(keys + i), "r"(kk[0]),
                     "r"(kk[1]), "r"(kk[2]), "r"(kk[3]), "l"(kpol) : "memory");
        // consecutive outputs often share the top digit: one atomic per run
        uint32_t bin = kk[0] >> 20, cnt = 1;
#pragma unroll
        for (int r = 1; r < 4; ++r) {
          const uint32_t br = kk[r] >> 20;
          if (br == bin) {
            ++cnt;
          } else {
            atomicAdd(&hist0[bin], cnt);
            bin = br;
            cnt = 1;
          }
        }
        atomicAdd(&hist0[bin], cnt);
      } else {
#pragma unroll
        for (int r = 0; r < 4; ++r)
          if (i + r >= 0 && i + r < Lc) {
            keys[i + r] = kk[r];
            atomicAdd(&hist0[kk[r] >> 20], 1u);
          }
      }
    };
    // two groups per pass: their loads are in flight together
    for (int q = tid; q < ngroups; q += 2 * NT) {
      float xm0[12], xs0[12], xm1[12], xs1[12];
      const bool two = q + NT < ngroups;
      load_group(q, xm0, xs0);
      if (two) load_group(q + NT, xm1, xs1);
      emit_group(q, xm0, xs0);
      if (two) emit_group(q + NT, xm1, xs1);
    }
  } else {
    // any other kernel: a tile holds kPoolRuns runs of kPoolRun consecutive outputs
    // per thread (run q of thread t starts at (q*NT + t)*kPoolRun)
    constexpr int kTile = NT * kPoolRun * kPoolRuns;
    const int tile_in = kTile + 2 * h;
    float* tsg = tmu + tile_in;
    // the loads of the next tile are in flight while this tile is pooled
    constexpr int kPer = (kTile + 2 * 127 + NT - 1) / NT;
    float lm[kPer], ls[kPer];
    auto load_tile = [&](int base) {
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        const int j = q * NT + tid;
        const int i = base - h + j;
        const bool in = (j < tile_in) && (i >= 0) && (i < Lc);
        lm[q] = in ? __ldg(mu + i) : -INFINITY;
        ls[q] = in ? __ldg(sg + i) : -INFINITY;
      }
    };
    load_tile(0);
    for (int base = 0; base < Lc; base += kTile) {
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        const int j = q * NT + tid;
        if (j < tile_in) {
          tmu[j] = lm[q];
          tsg[j] = ls[q];
        }
      }
      __syncthreads();
      if (base + kTile < Lc) load_tile(base + kTile);
#pragma unroll
      for (int q = 0; q < kPoolRuns; ++q) {
        const int o0 = (q * NT + tid) * kPoolRun;
        if (h <= 3) {
          // a 13-value window in registers covers the 7 outputs of the run for any
          // kernel up to 7; out[r] = max of x[o0+r .. o0+r+2h] (tile coordinates)
          float wm[kPoolRun + 6], ws[kPoolRun + 6];
#pragma unroll
          for (int j = 0; j < kPoolRun + 6; ++j) {
            const bool in = j < kPoolRun + 2 * h;
            wm[j] = in ? tmu[o0 + j] : -INFINITY;
            ws[j] = in ? tsg[o0 + j] : -INFINITY;
          }
#pragma unroll
          for (int r = 0; r < kPoolRun; ++r) {
            float mh = wm[r], shh = ws[r];
#pragma unroll
            for (int j = 1; j <= 6; ++j)
              if (j <= 2 * h) {
                mh = fmaxf(mh, wm[r + j]);
                shh = fmaxf(shh, ws[r + j]);
              }
            const int i = base + o0 + r;
            if (i < Lc) {
              const uint32_t k = ord_key(fmaf(lambda1, shh, mh));
              keys[i] = k;
              atomicAdd(&hist0[k >> 20], 1u);
            }
          }
        } else {
#pragma unroll
          for (int r = 0; r < kPoolRun; ++r) {
            const int i = base + o0 + r;
            if (i < Lc) {
              float mh = tmu[o0 + r], shh = tsg[o0 + r];
              for (int j = 1; j <= 2 * h; ++j) {
                mh = fmaxf(mh, tmu[o0 + r + j]);
                shh = fmaxf(shh, tsg[o0 + r + j]);
              }
              const uint32_t k = ord_key(fmaf(lambda1, shh, mh));
              keys[i] = k;
              atomicAdd(&hist0[k >> 20], 1u);
            }
          }
        }
      }
      __syncthreads();
    }
  }
  if (tid == 0) {
    sh.prefix = 0;
    sh.need = static_cast<uint32_t>(C);
    sh.cnt = 0;
    sh.maxkey = 0;
  }
  __syncthreads();

  // 2. radix select of the C-th largest key: digits of 12, 12 and 8 bits. The first
  //    digit's histogram came with the pooling; after it one scan sends every key
  //    above the threshold bin to the pool and copies the keys of that bin (key,
  //    position) to shared memory, where the two finer digits and the ties are
  //    resolved. A bin larger than the copy falls back to scans of the global keys.
  uint32_t* cand_k = reinterpret_cast<uint32_t*>(big + kBins * sizeof(uint32_t));
  int32_t* cand_p = reinterpret_cast<int32_t*>(cand_k + kCandCap<NT>());
  // histogram of the digit at `shift` over the keys matching the prefix, then the
  // digit where the count from the top first reaches `need`
  auto digit_pass = [&](int pass, uint32_t pmask, bool staged, uint32_t ncand) {
    const int shift = pass == 0 ? 20 : (pass == 1 ? 8 : 0);
    const int nb = pass == 2 ? 256 : kBins;
    uint32_t* hist = pass == 0 ? hist0 : hist12;
    if (pass > 0)
      for (int b = tid; b < nb; b += NT) hist[b] = 0;
    __syncthreads();
    const uint32_t prefix = sh.prefix;
    if (pass > 0 && staged) {
      for (uint32_t e = tid; e < ncand; e += NT) {
        const uint32_t k = cand_k[e];
        if ((k & pmask) == prefix) atomicAdd(&hist[(k >> shift) & static_cast<uint32_t>(nb - 1)], 1u);
      }
    }
    for (int i0 = 0; pass > 0 && !staged && i0 < Lc; i0 += NT * kBatch) {
      uint32_t kb[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        kb[j] = i < Lc ? __ldcg(&keys[i]) : 0u;
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        if ((i < Lc) && ((kb[j] & pmask) == prefix))
          atomicAdd(&hist[(kb[j] >> shift) & static_cast<uint32_t>(nb - 1)], 1u);
      }
    }
    __syncthreads();
    // thread t owns bins [t*per, (t+1)*per)
    const int per = nb / NT > 0 ? nb / NT : 1;
    const int b0 = tid * per;
    uint32_t mine = 0;
    if (b0 < nb)
      for (int b = 0; b < per; ++b) mine += hist[b0 + b];
    const uint32_t above = block_excl_suffix<NT>(mine, sh);
    const uint32_t need = sh.need;
    if (b0 < nb && above < need && above + mine >= need) {
      uint32_t acc = above;
      for (int b = per - 1; b >= 0; --b) {
        const uint32_t c = hist[b0 + b];
        if (acc + c >= need) {
          sh.prefix = prefix | (static_cast<uint32_t>(b0 + b) << shift);
          sh.need = need - acc;
          break;
        }
        acc += c;
      }
    }
    __syncthreads();
  };
  digit_pass(0, 0u, false, 0u);
  // the scan: keys above the first digit's bin go to the pool, that bin to `cand`
  if (tid == 0) {
    sh.cnt = 0;
    sh.ncand = 0;
  }
  __syncthreads();
  {
    const uint32_t bin = sh.prefix >> 20;
    for (int i0 = 0; i0 < Lc; i0 += NT * kBatch) {
      uint32_t kb[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        kb[j] = i < Lc ? __ldcg(&keys[i]) : 0u;
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        if (i < Lc) {
          const uint32_t d = kb[j] >> 20;
          if (d > bin) {
            const uint32_t e = atomicAdd(&sh.cnt, 1u);
            if (e < static_cast<uint32_t>(NT)) {   // always, unless the count check below fails
              cpos[e] = i;
              ckey[e] = kb[j];
            }
          } else if (d == bin) {
            const uint32_t e = atomicAdd(&sh.ncand, 1u);
            if (e < kCandCap<NT>()) {
              cand_k[e] = kb[j];
              cand_p[e] = i;
            }
          }
        }
      }
    }
  }
  __syncthreads();
  const uint32_t ncand = sh.ncand;
  const bool staged = ncand <= kCandCap<NT>();
  digit_pass(1, 0xFFFu << 20, staged, ncand);
  digit_pass(2, 0xFFFFFFu << 8, staged, ncand);
  const uint32_t T = sh.prefix;
  const uint32_t needT = sh.need;   // keys equal to T to take, lowest positions first

  // 3. every key above the threshold, and the positions of the keys equal to it
  //    (the tie list overlays the dead finer-digit histogram)
  int32_t* ties = reinterpret_cast<int32_t*>(big);   // [kTieCap]
  if (tid == 0) {
    sh.teq = 0;
    if (!staged) sh.cnt = 0;   // the global scans below collect the whole pool again
  }
  __syncthreads();
  if (staged) {
    for (uint32_t e = tid; e < ncand; e += NT) {
      const uint32_t k = cand_k[e];
      if (k > T) {
        const uint32_t n = atomicAdd(&sh.cnt, 1u);
        if (n < static_cast<uint32_t>(NT)) {
          cpos[n] = cand_p[e];
          ckey[n] = k;
        }
      } else if (k == T) {
        const uint32_t q = atomicAdd(&sh.teq, 1u);
        if (q < kTieCap) ties[q] = cand_p[e];
      }
    }
  } else {
    for (int i0 = 0; i0 < Lc; i0 += NT * kBatch) {
      uint32_t kb[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        kb[j] = i < Lc ? __ldcg(&keys[i]) : 0u;
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int i = i0 + j * NT + tid;
        if (i < Lc) {
          if (kb[j] > T) {
            const uint32_t n = atomicAdd(&sh.cnt, 1u);
            if (n < static_cast<uint32_t>(NT)) {
              cpos[n] = i;
              ckey[n] = kb[j];
            }
          } else if (kb[j] == T) {
            const uint32_t e = atomicAdd(&sh.teq, 1u);
            if (e < kTieCap) ties[e] = i;
          }
        }
      }
    }
  }
  __syncthreads();
  const uint32_t n_above = sh.cnt;
  const uint32_t n_eq = sh.teq;
  // Every path above leaves n_above = #{key > T} and n_eq = #{key == T} with
  // n_above + needT = C and needT <= n_eq, so that the ties below fill the pool to
  // exactly C positions (the pool writes above are bounded by the pool's size all the
  // same). Should that ever fail, the pool would hold unwritten slots: the unit is then
  // reported through the error word and gets no selection.
  if (n_above + needT != static_cast<uint32_t>(C) || needT > n_eq || needT == 0u) {
    if (tid == 0 && P.err) atomicOr(P.err, kErrCheck);
    int32_t* out = P.indices + out_off + u.unit * B;
    for (int r = tid; r < B; r += NT) out[r] = -1;
    if (P.order)
      for (int r = tid; r < B; r += NT) P.order[out_off + u.unit * B + r] = -1;
    if (P.margins)
      for (int r = tid; r < B; r += NT) P.margins[out_off + u.unit * B + r] = 0.f;
    if (P.k_out) write_compact_cache<NT>(P, u, Lc, nsel, 0, nullptr, nullptr, nullptr);
    return;
  }
  if (n_eq <= kTieCap) {
    // the needT lowest positions among the ties, by rank
    for (uint32_t e = tid; e < n_eq; e += NT) {
      const int pos = ties[e];
      uint32_t rank = 0;
      for (uint32_t f = 0; f < n_eq; ++f) rank += (ties[f] < pos);
      if (rank < needT) {
        cpos[n_above + rank] = pos;
        ckey[n_above + rank] = T;
      }
    }
  } else {
    // many equal keys: ordered block scan over the positions
    uint32_t taken = 0;
    for (int base = 0; base < Lc && taken < needT; base += NT) {
      const int i = base + tid;
      const bool f = (i < Lc) && (__ldcg(&keys[i]) == T);
      uint32_t tot;
      const uint32_t pre = block_excl_count<NT>(f, sh, &tot);
      if (f && taken + pre < needT) {
        cpos[n_above + taken + pre] = i;
        ckey[n_above + taken + pre] = T;
      }
      taken += tot;
    }
  }
  __syncthreads();

  // 4. the pool with its keys. Below 2^23 positions the greedy breaks ties by position
  //    itself (position and slot packed in 32 bits), so the pool stays in the order it
  //    was collected in; beyond that the pool is sorted by position, so that "lower
  //    slot" means "lower position". Normalise, stage keys and inverse norms.
  const bool packed = Lc < (1 << 23);   // position << 9 | slot stays below 0xFFFFFFFF
  const int32_t* ppos = packed ? cpos : spos;
  const uint32_t* pkey = packed ? ckey : skey;
  if (tid < C) {
    const int pos = cpos[tid];
    const uint32_t key = ckey[tid];
    if (!packed) {
      int rank = 0;
      for (int c = 0; c < C; ++c) rank += (cpos[c] < pos);
      spos[rank] = pos;
      skey[rank] = key;
    }
    atomicMax(&sh.maxkey, key);
  }
  __syncthreads();
  const float smax = fmaxf(unord_key(sh.maxkey), P.norm_eps);
  // candidate keys row-major in shared memory; a half-warp copies one 256-byte row,
  // coalesced
  {
    constexpr int kRows = NT / (NT / 32 * 2);      // rows per half-warp: 8 (NT=256) or 16 (NT=512)
    uint4 xr[kRows];
#pragma unroll
    for (int q = 0; q < kRows; ++q) {
      const int r = (q * (NT / 32) + warp) * 2 + (lane >> 4);
      xr[q] = make_uint4(0, 0, 0, 0);
      if (r < C) {
        const int pos = ppos[r];
        if (pos >= 0 && pos < Lc) {
          const uint4* src = reinterpret_cast<const uint4*>(P.k + u.k_off + pos * P.g.k_st);
          xr[q] = __ldg(src + (lane & 15));
        } else if (P.err) {
          atomicOr(P.err, kErrCheck);   // never read outside the unit's keys
        }
      }
    }
#pragma unroll
    for (int q = 0; q < kRows; ++q) {
      const int r = (q * (NT / 32) + warp) * 2 + (lane >> 4);
      if (r < C) krow[r * kRowChunks + (lane & 15)] = xr[q];
    }
  }
  __syncthreads();

  // 5. greedy admissions. Lane (g, t) of a warp owns slot
  //    warp*32 + 16*(t>>1) + g + 8*(t&1); the warp's 32 candidate keys stay in
  //    registers as mma.m16n8k16 A fragments, and every admission computes the
  //    32 dot products with the admitted key by 16 tensor-core MMAs (bf16 products,
  //    fp32 accumulation) with that key replicated in the 8 columns of B. The
  //    argmax takes the largest value, then the smallest tie key (position << 9 |
  //    slot, or the slot of a sorted pool): ties go to the lower position.
  const int g = lane >> 2, tq = lane & 3;
  const int slot = warp * 32 + 16 * (tq >> 1) + g + 8 * (tq & 1);
  bool active = slot < C;
  float corr = 0.f;
  const float my_st = active ? __fdiv_rn(unord_key(pkey[slot]), smax) : 0.f;
  // the candidate's inverse norm, from its own staged row (the admitted key's comes
  // from inv[] after the first barrier of the loop below)
  float my_inv = 0.f;
  if (active) {
    const uint4* row = krow + slot * kRowChunks;
    float ss0 = 0.f, ss1 = 0.f;
#pragma unroll 4
    for (int c = 0; c < kChunks; ++c) {
      const uint4 w = row[c];
      const uint32_t w4[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float lo = __uint_as_float(w4[e] << 16);
        const float hi = __uint_as_float(w4[e] & 0xFFFF0000u);
        ss0 = fmaf(lo, lo, ss0);
        ss1 = fmaf(hi, hi, ss1);
      }
    }
    const float ss = ss0 + ss1;
    my_inv = ss > 0.f ? inv_sqrt(ss) : 0.f;
    inv[slot] = my_inv;
  }
  const uint32_t my_tie = !active ? 0xFFFFFFFFu
                                  : (packed ? (static_cast<uint32_t>(ppos[slot]) << 9) | static_cast<uint32_t>(slot)
                                            : static_cast<uint32_t>(slot));
  const uint32_t* kw = reinterpret_cast<const uint32_t*>(krow);   // 4 * kRowChunks words per row
  uint32_t afr[2][8][4];
#pragma unroll
  for (int m = 0; m < 2; ++m) {
    const int r0 = warp * 32 + 16 * m + g, r1 = r0 + 8;
#pragma unroll
    for (int s8 = 0; s8 < 8; ++s8) {
      afr[m][s8][0] = r0 < C ? kw[r0 * kRowWords + 8 * s8 + tq] : 0u;
      afr[m][s8][1] = r1 < C ? kw[r1 * kRowWords + 8 * s8 + tq] : 0u;
      afr[m][s8][2] = r0 < C ? kw[r0 * kRowWords + 8 * s8 + tq + 4] : 0u;
      afr[m][s8][3] = r1 < C ? kw[r1 * kRowWords + 8 * s8 + tq + 4] : 0u;
    }
  }
  int32_t* order = P.order ? P.order + out_off + u.unit * B : nullptr;
  float* margins = P.margins ? P.margins + out_off + u.unit * B : nullptr;
  // admitted positions in admission order (the pool's other pair of arrays is free),
  // and their slots when the compact cache is written here
  int32_t* adm = packed ? spos : cpos;
  int32_t* adm_slot = reinterpret_cast<int32_t*>(packed ? skey : ckey);
  for (int t = 0; t < nsel; ++t) {
    const uint32_t key = active ? ord_key(fmaf(lambda2, corr, my_st)) : 0u;
    const uint32_t wmax = __reduce_max_sync(0xffffffffu, key);
    const uint32_t wtie = __reduce_min_sync(0xffffffffu, (active && key == wmax) ? my_tie : 0xFFFFFFFFu);
    // the runner-up only feeds the margins output
    const uint32_t wsec = margins ? __reduce_max_sync(0xffffffffu, my_tie == wtie ? 0u : key) : 0u;
    if (lane == 0) {
      sh.red[t & 1][warp][0] = wmax;
      sh.red[t & 1][warp][1] = wtie;
      sh.red[t & 1][warp][2] = wsec;
    }
    __syncthreads();
    // every warp reduces the NT/32 warp results itself (lane w holds warp w's)
    const bool hold = lane < NT / 32;
    const uint32_t k_l = hold ? sh.red[t & 1][lane][0] : 0u;
    const uint32_t tie_l = hold ? sh.red[t & 1][lane][1] : 0xFFFFFFFFu;
    const uint32_t best = __reduce_max_sync(0xffffffffu, k_l);
    const uint32_t btie = __reduce_min_sync(0xffffffffu, k_l == best ? tie_l : 0xFFFFFFFFu);
    uint32_t sec = 0;
    if (margins) {
      const uint32_t k2_l = hold ? sh.red[t & 1][lane][2] : 0u;
      // runner-up: the other warps' best and the winning warp's second
      sec = __reduce_max_sync(0xffffffffu, (k_l == best && tie_l == btie) ? k2_l : max(k_l, k2_l));
    }
    const int js = static_cast<int>(packed ? (btie & 511u) : btie);
    if (tid == 0) {
      const int pos = packed ? static_cast<int>(btie >> 9) : ppos[js];
      adm[t] = pos;
      adm_slot[t] = js;
      if (order) order[t] = pos;
      if (margins) margins[t] = sec ? unord_key(best) - unord_key(sec) : INFINITY;
    }
    if (slot == js) active = false;
    // dots of the warp's candidates with the admitted key (four accumulation chains
    // per tile: k-steps modulo 4)
    float d[2][4][4];
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int e = 0; e < 4; ++e) d[m][c][e] = 0.f;
    uint32_t bf[8][2];
#pragma unroll
    for (int s8 = 0; s8 < 8; ++s8) {
      bf[s8][0] = kw[js * kRowWords + 8 * s8 + tq];
      bf[s8][1] = kw[js * kRowWords + 8 * s8 + tq + 4];
    }
#pragma unroll
    for (int s8 = 0; s8 < 8; ++s8) {
#pragma unroll
      for (int m = 0; m < 2; ++m) {
        float* dd = d[m][s8 & 3];
        asm volatile(
            "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
            "{%8,%9}, {%0,%1,%2,%3};"
            : "+f"(dd[0]), "+f"(dd[1]), "+f"(dd[2]), "+f"(dd[3])
            : "r"(afr[m][s8][0]), "r"(afr[m][s8][1]), "r"(afr[m][s8][2]), "r"(afr[m][s8][3]),
              "r"(bf[s8][0]), "r"(bf[s8][1]));
      }
    }
    // rows g (element 0) and g + 8 (element 2) of tile t>>1; every column holds the same dot
    // (register-only selection: no runtime index into d)
    float dm[2][2];
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
      for (int e = 0; e < 2; ++e)
        dm[m][e] = (d[m][0][2 * e] + d[m][1][2 * e]) + (d[m][2][2 * e] + d[m][3][2 * e]);
    const float dlo = (tq & 1) ? dm[0][1] : dm[0][0];
    const float dhi = (tq & 1) ? dm[1][1] : dm[1][0];
    const float dot = (tq >> 1) ? dhi : dlo;
    if (active) corr = fmaxf(corr, dot * my_inv * inv[js]);
  }

  // 6. admitted positions in ascending order (rank among the nsel admissions), then -1
  __syncthreads();
  int32_t* out = P.indices + out_off + u.unit * B;
  // (with the compact cache: position and staged row by rank, where the first-digit
  // histogram was)
  int32_t* rpos = reinterpret_cast<int32_t*>(hist0);
  int32_t* rslot = rpos + kMaxPoolCand;   // ranks < nsel <= C <= kMaxPoolCand
  for (int e = tid; e < nsel; e += NT) {
    const int pos = adm[e];
    int rank = 0;
    for (int f = 0; f < nsel; ++f) rank += (adm[f] < pos);
    out[rank] = pos;
    if (P.k_out) {
      rpos[rank] = pos;
      rslot[rank] = adm_slot[e];
    }
  }
  for (int r = nsel + tid; r < B; r += NT) out[r] = -1;
  if (order)
    for (int r = nsel + tid; r < B; r += NT) order[r] = -1;
  if (margins)
    for (int r = nsel + tid; r < B; r += NT) margins[r] = 0.f;
  if (P.k_out) {
    __syncthreads();
    write_compact_cache<NT>(P, u, Lc, nsel, nsel, rpos, rslot, krow);
  }
}

template <int NT>
constexpr size_t select_smem() {
  // candidate keys (also reused for the pooling tiles, the histograms, the threshold
  // bin's keys and the tie list) + 5 arrays + the first-digit histogram
  return kRowChunks * NT * sizeof(uint4) + 5 * NT * sizeof(int32_t) + kBins * sizeof(uint32_t);
}
static_assert(kRowChunks * 256 * sizeof(uint4) >= kBins * sizeof(uint32_t), "histogram fits");
static_assert(kRowChunks * 256 * sizeof(uint4) >= 2 * (256 * kPoolRun * kPoolRuns + 256) * sizeof(float),
              "pool tiles fit");
static_assert(kRowChunks * 256 * sizeof(uint4) >= kTieCap * sizeof(int32_t), "tie list fits");
static_assert(2 * kMaxPoolCand <= kBins, "ranked positions and rows fit the first-digit histogram's place");
// both parameter blocks of a multi-profile launch fit the 32764-byte kernel
// parameter space
static_assert(sizeof(SelectParams) + sizeof(ProfileTable) + 64 <= 32764, "profile table fits");

}  // namespace

template <class Prof>
cudaError_t launch_select_grid(const kve_plan& plan, const SelectParams& p, const Prof& prof,
                               unsigned profiles, cudaStream_t stream) {
  // pool size bound: the largest C over the requests
  int max_lc = 0;
  for (int r = 0; r < plan.geo.n_req; ++r) max_lc = max(max_lc, plan.geo.req_len[r] - plan.geo.window);
  const int cmax = p.cand_factor == 0 ? max_lc : min(p.cand_factor * p.budget, max_lc);
  const dim3 grid(static_cast<unsigned>(plan.geo.n_units), profiles);
  if (cmax <= 256) {
    constexpr size_t smem = select_smem<256>();
    cudaError_t e = cudaFuncSetAttribute(select_kernel<256, Prof>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    return launch_after_previous(select_kernel<256, Prof>, grid, dim3(256), smem, stream, p, prof);
  } else {
    constexpr size_t smem = select_smem<512>();
    cudaError_t e = cudaFuncSetAttribute(select_kernel<512, Prof>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    return launch_after_previous(select_kernel<512, Prof>, grid, dim3(512), smem, stream, p, prof);
  }
}

cudaError_t launch_select(const kve_plan& plan, const SelectParams& p, cudaStream_t stream) {
  return launch_select_grid(plan, p, OneProfile{}, 1u, stream);
}

cudaError_t launch_select_profiles(const kve_plan& plan, const SelectParams& p, const ProfileTable& table,
                                   int profiles, cudaStream_t stream) {
  return launch_select_grid(plan, p, table, static_cast<unsigned>(profiles), stream);
}

}  // namespace kve

// ---------------------------------------------------------------------------
// Selection without caller-provided scratch.
//
// Some callers cannot allocate device memory when they evict: serving engines
// that reserve nearly all of HBM up front for their own KV-cache pool and hand
// kernels nothing but pointers into it (a cudaMalloc there fails or breaks the
// engine's accounting, and it also synchronises the device), or plugin hosts that
// give a kernel only its input and output buffers. For them the select kernel's
// one scratch buffer -- the ordered base score of every candidate token -- lives
// in a fixed array compiled into this library.
namespace kve {
namespace {

constexpr size_t kNoAllocScratchWords = size_t(4) << 20;   // 16 MiB of uint32 keys

// Reserved on every GPU that loads the library, for the life of the process.
static __device__ __align__(256) uint32_t g_select_scratch[kNoAllocScratchWords];
// Its error word (the workspace's first word plays this part for the other entry
// points); zero at load, read and cleared by kv_evict_status with ws = NULL.
static __device__ __align__(256) uint32_t g_noalloc_err;

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
uint32_t* g_scratch_ptr[kMaxDevices] = {};
uint32_t* g_err_ptr[kMaxDevices] = {};

// Device addresses of g_select_scratch and g_noalloc_err on the current device
// (looked up once per device; in host code the symbols themselves are only host-side
// stand-ins). False when the lookup fails.
bool noalloc_addresses(uint32_t** scratch, uint32_t** err) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    void* e = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_scratch) != cudaSuccess) return false;
    if (cudaGetSymbolAddress(&e, g_noalloc_err) != cudaSuccess) return false;
    g_err_ptr[dev] = static_cast<uint32_t*>(e);
    g_scratch_ptr[dev] = static_cast<uint32_t*>(p);
  }
  *scratch = g_scratch_ptr[dev];
  *err = g_err_ptr[dev];
  return true;
}

}  // namespace

uint32_t* noalloc_error_word() {
  uint32_t *scratch = nullptr, *err = nullptr;
  return noalloc_addresses(&scratch, &err) ? err : nullptr;
}

}  // namespace kve

extern "C" kve_status kv_evict_select_noalloc(const kve_plan* plan, const float* mu, const float* sigma,
                                              const uint16_t* k, const float* lambda1,
                                              const float* lambda2, int32_t* indices, int32_t* order,
                                              float* margins, void* stream) {
  using namespace kve;
  if (!plan || !mu || !sigma || !k || !lambda1 || !lambda2 || !indices || plan->select_all)
    return KVE_EINVAL;
  const Geometry& g = plan->geo;
  // one scratch word per prefix token of every unit: N_L x (units per layer) x SL
  const size_t words = static_cast<size_t>(g.num_layers) * g.uheads * static_cast<size_t>(g.total_tokens);
  if (words > kNoAllocScratchWords) return KVE_EINVAL;   // beyond the fixed scratch
  if (((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(mu) |
        reinterpret_cast<uintptr_t>(sigma)) & 15u) != 0)
    return KVE_EINVAL;   // the header asks every pointer to be 16-byte aligned
  SelectParams p;
  const kve_status s = select_params(plan, mu, sigma, k, lambda1, lambda2, indices, order, margins, &p);
  if (s != KVE_OK) return s;
  if (!noalloc_addresses(&p.keys, &p.err)) return KVE_ECUDA;
  return launch_select(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK : KVE_ECUDA;
}
