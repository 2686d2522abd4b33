// Selector over every candidate (candidate_factor = 0 with Lc above the pooled
// selector's 512-slot pool): step 3 of the eviction step with C = Lc, one CTA per
// unit. Section 3.2 restricts the greedy to the top 4B tokens for speed; this path
// is the unrestricted ablation and admits exactly what the full greedy of Eq. 5
// admits over all Lc candidates.
//
//  1. max-pool mu and sigma over 0 .. Lc-1 (odd kernel, window clipped to the
//     range) and form s_i = mu_i + lambda1 sigma_i; s~ = s / max(max s, eps);
//  2. greedy admissions by s~_i + lambda2 corr_i, ties to the lower position, with
//     corr_i = max over admitted j of cos(k_i, k_j) (clamped at 0 by starting at 0).
//     With lambda2 <= 0 a value can only fall as the admitted set grows, so a value
//     computed against fewer admitted keys is an upper bound: each step takes the
//     best value; if it is stale, every thread whose own best candidate is stale
//     brings that candidate up to date (in parallel) and the search repeats; a
//     candidate whose value is current when it is the best is the full greedy's
//     choice (any candidate with an equal bound has a higher position).
//     With lambda2 > 0 every candidate is brought up to date after each admission.
//     When margins are requested the runner-up is brought up to date the same way.
//  3. write the admitted positions ascending (and in admission order, with margins).
// Values live in shared memory (C <= 32768); s~, corr and the inverse key norms in
// the workspace; the first 96 admitted keys are staged in shared memory, later ones
// are read from K in global memory (L2). For lambda2 <= 0 a warp refreshes its lanes'
// stale bests together on the tensor cores; for lambda2 > 0 a thread applies the
// missing admissions in groups of eight per pass over the candidate's row.
#include "kve_internal.h"

namespace kve {
namespace {

constexpr int kAllThreads = 1024;
constexpr int kAllWarps = kAllThreads / 32;
constexpr int kAdmStage = 96;          // admitted keys staged in shared memory
constexpr int kAdmStride = 17;         // uint4 per staged row (16 + 1 against bank conflicts)
constexpr int kRefreshGroup = 8;       // missing admissions applied per pass over a candidate row

__device__ __forceinline__ uint32_t ord_key_all(float f) {
  const uint32_t u = __float_as_uint(f + 0.0f);   // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

struct AllSmall {
  uint32_t wkey[kAllWarps];
  uint32_t widx[kAllWarps];
  float wmax[kAllWarps];
  uint32_t best_key, best_idx;
};

// Block argmax of the owners' bests: the largest key, ties to the lowest index.
__device__ __forceinline__ void block_best(uint32_t key, uint32_t idx, AllSmall& sh) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t wk = __reduce_max_sync(0xffffffffu, key);
  const uint32_t wi = __reduce_min_sync(0xffffffffu, key == wk ? idx : 0xFFFFFFFFu);
  if (lane == 0) {
    sh.wkey[warp] = wk;
    sh.widx[warp] = wi;
  }
  __syncthreads();
  if (warp == 0) {
    const uint32_t k = sh.wkey[lane], i = sh.widx[lane];
    const uint32_t bk = __reduce_max_sync(0xffffffffu, k);
    const uint32_t bi = __reduce_min_sync(0xffffffffu, k == bk ? i : 0xFFFFFFFFu);
    if (lane == 0) {
      sh.best_key = bk;
      sh.best_idx = bi;
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kAllThreads, 1) select_all_kernel(const __grid_constant__ SelectParams P) {
  wait_previous_kernel();   // mu and sigma come from the score kernel launched before
  __shared__ AllSmall sh;
  extern __shared__ __align__(16) uint8_t dyn[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  const UnitInfo u = unit_info(P.g, blockIdx.x);
  const int W = P.g.window;
  const int C = u.L - W;                      // every candidate
  const int B = P.budget;
  const int Bl = P.layer_budget[u.layer];
  const int nsel = min(Bl, C);
  const float lambda1 = P.lambda1[u.layer];
  const float lambda2 = P.lambda2[u.layer];
  const bool lazy = !(lambda2 > 0.f);
  const float* mu = P.mu + u.mu_off;
  const float* sg = P.sigma + u.mu_off;
  float* st = reinterpret_cast<float*>(P.keys + u.mu_off);   // s~ per candidate
  float2* cinv = reinterpret_cast<float2*>(P.corr) + u.mu_off;   // (corr_i, 1 / |k_i|)
  const uint16_t* kb = P.k + u.k_off;   // key i at kb + i * k_st
  const int64_t kst = P.g.k_st;
  const int h = P.pool_kernel / 2;

  float* v = reinterpret_cast<float*>(dyn);                         // [kMaxAllCand]
  uint16_t* applied = reinterpret_cast<uint16_t*>(v + kMaxAllCand);  // [kMaxAllCand]
  int32_t* adm = reinterpret_cast<int32_t*>(applied + kMaxAllCand);  // [kMaxAllBudget]
  float* adm_inv = reinterpret_cast<float*>(adm + kMaxAllBudget);    // [kMaxAllBudget]
  uint4* admk = reinterpret_cast<uint4*>(adm_inv + kMaxAllBudget);    // [kAdmStage][kAdmStride]

  // 1. pooled base score and its maximum
  float lmax = -INFINITY;
  for (int i = tid; i < C; i += kAllThreads) {
    const int a = max(i - h, 0), b = min(i + h, C - 1);
    float mh = -INFINITY, shh = -INFINITY;
    for (int j = a; j <= b; ++j) {
      mh = fmaxf(mh, __ldg(mu + j));
      shh = fmaxf(shh, __ldg(sg + j));
    }
    const float s = fmaf(lambda1, shh, mh);
    st[i] = s;
    lmax = fmaxf(lmax, s);
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
  if (lane == 0) sh.wmax[warp] = lmax;
  __syncthreads();
  float smax = sh.wmax[0];
  for (int w = 1; w < kAllWarps; ++w) smax = fmaxf(smax, sh.wmax[w]);
  smax = fmaxf(smax, P.norm_eps);
  for (int i = tid; i < C; i += kAllThreads) {
    const float s = __fdiv_rn(st[i], smax);
    st[i] = s;
    v[i] = s;                     // corr = 0: s~ + lambda2 * 0
    applied[i] = 0;
    const uint4* ki = reinterpret_cast<const uint4*>(kb + static_cast<int64_t>(i) * kst);
    float ss = 0.f;
    for (int c = 0; c < kHeadDim / 8; ++c) {
      const uint4 x = __ldg(ki + c);
      const uint32_t w4[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        ss = fmaf(bf16_lo(w4[e]), bf16_lo(w4[e]), ss);
        ss = fmaf(bf16_hi(w4[e]), bf16_hi(w4[e]), ss);
      }
    }
    cinv[i] = make_float2(0.f, ss > 0.f ? __fdiv_rn(1.0f, sqrtf(ss)) : 0.f);
  }
  __syncthreads();

  // the owner of candidate i is thread i % kAllThreads; it keeps the best of its own
  uint32_t my_key = 0, my_idx = 0xFFFFFFFFu;
  auto rescan = [&]() {
    my_key = 0;
    my_idx = 0xFFFFFFFFu;
    for (int i = tid; i < C; i += kAllThreads) {
      const float x = v[i];
      if (x == -INFINITY) continue;   // admitted
      const uint32_t k = ord_key_all(x);
      if (k > my_key || my_idx == 0xFFFFFFFFu) {
        my_key = k;
        my_idx = static_cast<uint32_t>(i);
      }
    }
  };
  rescan();

  // candidate i brought up to date with admissions applied[i] .. t-1 by its owner,
  // kRefreshGroup admissions per pass over the candidate's row (each dot keeps the
  // element order of a plain loop); staged admitted keys come from shared memory
  auto refresh = [&](int i, int t) {
    const uint4* ki = reinterpret_cast<const uint4*>(kb + static_cast<int64_t>(i) * kst);
    const float2 ci = cinv[i];
    const float inv_i = ci.y;
    float cmax = ci.x;
    // admitted key a, chunk c: staged in shared memory or read from K
    auto adm_chunk = [&](int a, int c) -> uint4 {
      return a < kAdmStage ? admk[a * kAdmStride + c]
                           : __ldg(reinterpret_cast<const uint4*>(kb + static_cast<int64_t>(adm[a]) * kst) + c);
    };
    int a0 = applied[i];
    for (; a0 + kRefreshGroup <= t; a0 += kRefreshGroup) {
      float dot[kRefreshGroup];
#pragma unroll
      for (int q = 0; q < kRefreshGroup; ++q) dot[q] = 0.f;
      for (int c = 0; c < kHeadDim / 8; ++c) {
        const uint4 x = __ldg(ki + c);
        const uint32_t xa[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int q = 0; q < kRefreshGroup; ++q) {
          const uint4 y = adm_chunk(a0 + q, c);
          const uint32_t ya[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            dot[q] = fmaf(bf16_lo(xa[e]), bf16_lo(ya[e]), dot[q]);
            dot[q] = fmaf(bf16_hi(xa[e]), bf16_hi(ya[e]), dot[q]);
          }
        }
      }
#pragma unroll
      for (int q = 0; q < kRefreshGroup; ++q) cmax = fmaxf(cmax, dot[q] * inv_i * adm_inv[a0 + q]);
    }
    for (; a0 < t; ++a0) {
      float dot = 0.f;
      for (int c = 0; c < kHeadDim / 8; ++c) {
        const uint4 x = __ldg(ki + c), y = adm_chunk(a0, c);
        const uint32_t xa[4] = {x.x, x.y, x.z, x.w}, ya[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          dot = fmaf(bf16_lo(xa[e]), bf16_lo(ya[e]), dot);
          dot = fmaf(bf16_hi(xa[e]), bf16_hi(ya[e]), dot);
        }
      }
      cmax = fmaxf(cmax, dot * inv_i * adm_inv[a0]);
    }
    cinv[i] = make_float2(cmax, inv_i);
    v[i] = fmaf(lambda2, cmax, st[i]);
    applied[i] = static_cast<uint16_t>(t);
  };
  // every owner whose best is stale brings it up to date, then takes its new best.
  // A warp refreshes its lanes' stale bests together on the tensor cores: lane r's
  // candidate row is row r of the A operand of mma.m16n8k16 (two m-tiles), the
  // admitted keys a_lo .. t-1 form the B operand, 16 per pass (two n-tiles), where
  // a_lo is the smallest count applied among the warp's stale bests; a dot against
  // an admission already applied leaves the running maximum unchanged.
  const uint32_t* kw32 = reinterpret_cast<const uint32_t*>(kb);          // row i at kw32 + i * kst / 2
  const int64_t kst32 = kst / 2;
  const uint32_t* admw = reinterpret_cast<const uint32_t*>(admk);        // 4 * kAdmStride words per row
  auto refresh_stale_bests = [&](int t) {
    const bool stale = my_idx != 0xFFFFFFFFu && applied[my_idx] < t;
    if (__any_sync(0xffffffffu, stale)) {
      const int a_lo = static_cast<int>(__reduce_min_sync(
          0xffffffffu, stale ? static_cast<uint32_t>(applied[my_idx]) : static_cast<uint32_t>(t)));
      const int row = stale ? static_cast<int>(my_idx) : 0;      // row 0: a valid stand-in
      const float2 ci = stale ? cinv[my_idx] : make_float2(0.f, 0.f);
      float cm = ci.x;
      const int g = lane >> 2, tq = lane & 3;
      // rows g and g + 8 of m-tiles 0 and 1 belong to lanes 16m + 8hh + g
      const uint32_t* ra[2][2];
      float ir[2][2];
#pragma unroll
      for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int src = 16 * m + 8 * hh + g;
          ra[m][hh] = kw32 + static_cast<int64_t>(__shfl_sync(0xffffffffu, row, src)) * kst32;
          ir[m][hh] = __shfl_sync(0xffffffffu, ci.y, src);
        }
      for (int a0 = a_lo; a0 < t; a0 += 16) {
        float d[2][2][4];
#pragma unroll
        for (int m = 0; m < 2; ++m)
#pragma unroll
          for (int n = 0; n < 2; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) d[m][n][e] = 0.f;
        // column g of n-tile n is admission a0 + 8n + g (zero past t)
        const uint32_t* rb[2];
        bool bv[2];
#pragma unroll
        for (int n = 0; n < 2; ++n) {
          const int an = a0 + 8 * n + g;
          bv[n] = an < t;
          rb[n] = !bv[n] ? kw32
                         : (an < kAdmStage ? admw + an * (4 * kAdmStride)
                                           : kw32 + static_cast<int64_t>(adm[an]) * kst32);
        }
#pragma unroll
        for (int s8 = 0; s8 < kHeadDim / 16; ++s8) {
          uint32_t af[2][4];
#pragma unroll
          for (int m = 0; m < 2; ++m) {
            af[m][0] = __ldg(ra[m][0] + 8 * s8 + tq);
            af[m][1] = __ldg(ra[m][1] + 8 * s8 + tq);
            af[m][2] = __ldg(ra[m][0] + 8 * s8 + tq + 4);
            af[m][3] = __ldg(ra[m][1] + 8 * s8 + tq + 4);
          }
#pragma unroll
          for (int n = 0; n < 2; ++n) {
            const uint32_t b0 = bv[n] ? rb[n][8 * s8 + tq] : 0u;
            const uint32_t b1 = bv[n] ? rb[n][8 * s8 + tq + 4] : 0u;
#pragma unroll
            for (int m = 0; m < 2; ++m) {
              float* dd = d[m][n];
              asm volatile(
                  "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
                  "{%8,%9}, {%0,%1,%2,%3};"
                  : "+f"(dd[0]), "+f"(dd[1]), "+f"(dd[2]), "+f"(dd[3])
                  : "r"(af[m][0]), "r"(af[m][1]), "r"(af[m][2]), "r"(af[m][3]), "r"(b0), "r"(b1));
            }
          }
        }
        // element 2hh + e of d[m][n] is (row g + 8hh of m-tile m, column 2tq + e)
        float rmax[2][2];
#pragma unroll
        for (int m = 0; m < 2; ++m) rmax[m][0] = rmax[m][1] = -INFINITY;
#pragma unroll
        for (int n = 0; n < 2; ++n)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int a = a0 + 8 * n + 2 * tq + e;
            if (a < t) {
              const float ia = adm_inv[a];
#pragma unroll
              for (int m = 0; m < 2; ++m)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh)
                  rmax[m][hh] = fmaxf(rmax[m][hh], d[m][n][2 * hh + e] * ir[m][hh] * ia);
            }
          }
#pragma unroll
        for (int m = 0; m < 2; ++m)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            rmax[m][hh] = fmaxf(rmax[m][hh], __shfl_xor_sync(0xffffffffu, rmax[m][hh], 1));
            rmax[m][hh] = fmaxf(rmax[m][hh], __shfl_xor_sync(0xffffffffu, rmax[m][hh], 2));
          }
        // lane 16m + 8hh + gg takes row (m, gg + 8hh) from lane 4gg
        const int src = 4 * (lane & 7);
        const float r00 = __shfl_sync(0xffffffffu, rmax[0][0], src);
        const float r01 = __shfl_sync(0xffffffffu, rmax[0][1], src);
        const float r10 = __shfl_sync(0xffffffffu, rmax[1][0], src);
        const float r11 = __shfl_sync(0xffffffffu, rmax[1][1], src);
        const float mine = (lane >> 4) ? ((lane >> 3) & 1 ? r11 : r10) : ((lane >> 3) & 1 ? r01 : r00);
        cm = fmaxf(cm, mine);
      }
      if (stale) {
        cinv[my_idx] = make_float2(cm, ci.y);
        v[my_idx] = fmaf(lambda2, cm, st[my_idx]);
        applied[my_idx] = static_cast<uint16_t>(t);
        rescan();
      }
    }
    __syncthreads();
  };

  int32_t* order = P.order ? P.order + u.unit * B : nullptr;
  float* margins = P.margins ? P.margins + u.unit * B : nullptr;
  int t = 0;
  while (t < nsel) {
    block_best(my_key, my_idx, sh);
    const int bi = static_cast<int>(sh.best_idx);
    if (applied[bi] < t) {            // a stale bound: bring stale bests up to date, search again
      refresh_stale_bests(t);
      continue;
    }
    // bi is the full greedy's admission at step t
    const float vstar = v[bi];
    __syncthreads();                  // every thread has read v[bi] and applied[bi]
    if (tid == 0) {
      adm[t] = bi;
      v[bi] = -INFINITY;
      if (order) order[t] = bi;
    }
    if (t < kAdmStage && tid < kHeadDim / 8)
      admk[t * kAdmStride + tid] =
          __ldg(reinterpret_cast<const uint4*>(kb + static_cast<int64_t>(bi) * kst) + tid);
    __syncthreads();
    if (tid == (bi % kAllThreads)) rescan();
    if (margins) {
      // the runner-up, brought up to date against admissions 0 .. t-1
      for (;;) {
        block_best(my_key, my_idx, sh);
        const uint32_t si = sh.best_idx;
        if (si == 0xFFFFFFFFu) {
          if (tid == 0) margins[t] = INFINITY;
          break;
        }
        if (applied[si] < t) {
          refresh_stale_bests(t);
          continue;
        }
        if (tid == 0) margins[t] = vstar - v[si];
        break;
      }
    }
    if (tid == 0) adm_inv[t] = cinv[bi].y;   // inverse norm of the admitted key
    __syncthreads();
    ++t;
    if (!lazy && t < nsel) {
      // lambda2 > 0: values grow with corr, so every candidate is brought up to date
      for (int i = tid; i < C; i += kAllThreads)
        if (v[i] != -INFINITY) refresh(i, t);
      __syncthreads();
      rescan();
    }
  }

  // 3. admitted positions ascending, then -1: entry a of the admission order goes to
  //    its rank among the admitted positions (all distinct); nsel <= kMaxAllBudget
  __syncthreads();
  int32_t* out = P.indices + u.unit * B;
  for (int a = tid; a < nsel; a += kAllThreads) {
    const int pos = adm[a];
    int rank = 0;
    for (int c = 0; c < nsel; ++c) rank += (adm[c] < pos);
    out[rank] = pos;
  }
  for (int r = nsel + tid; r < B; r += kAllThreads) out[r] = -1;
  if (order)
    for (int r = nsel + tid; r < B; r += kAllThreads) order[r] = -1;
  if (margins)
    for (int r = nsel + tid; r < B; r += kAllThreads) margins[r] = 0.f;
}

}  // namespace

cudaError_t launch_select_all(const kve_plan& plan, const SelectParams& p, cudaStream_t stream) {
  constexpr size_t smem = kMaxAllCand * (sizeof(float) + sizeof(uint16_t)) +
                          kMaxAllBudget * (sizeof(int32_t) + sizeof(float)) +
                          kAdmStage * kAdmStride * sizeof(uint4);
  cudaError_t e = cudaFuncSetAttribute(select_all_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch_after_previous(select_all_kernel, dim3(static_cast<unsigned>(plan.geo.n_units)),
                               dim3(kAllThreads), smem, stream, p);
}

}  // namespace kve
