// Selector kernel: step 3 of the eviction step, one CTA per unit.
//
//  1. max-pool mu and sigma over the candidate tokens 0 .. Lc-1 (Section 3.1 keeps
//     the baselines' pooling; odd kernel, stride 1, window clipped to the range)
//     and form the base score s_i = mu_i + lambda1 sigma_i (Eq. 2 without corr);
//     s is stored as an order-preserving 32-bit key in the workspace;
//  2. find the C = min(factor*B, Lc) largest keys (Section 3.2: the greedy runs on
//     the top 4B tokens) by an MSB-first radix select; ties at the cut go to the
//     lower positions;
//  3. normalise s~ = s / max(max s, eps) (Eq. 5) and stage the candidate keys
//     (bf16) and their inverse norms in shared memory, candidates sorted by
//     position so that "lower slot" means "lower position";
//  4. admit min(B, C) candidates greedily (Eq. 5): value s~ + lambda2 corr, ties to
//     the lower position; after every admission j, corr_i <- max(corr_i,
//     cos(k_i, k_j)), which is Eq. 4 for the grown set (corr starts at 0, which is
//     both corr(i, {}) and the clamp at 0);
//  5. write the admitted positions ascending (and optionally in admission order,
//     with the best-minus-second margin of every admission).
#include <mutex>

#include "kve_internal.h"

namespace kve {
namespace {

constexpr int kSelThreads = 512;
constexpr int kMaxCand = 512;
constexpr int kChunks = kHeadDim / 8;   // 16-byte chunks of a key row

__device__ __forceinline__ uint32_t ord_key(float f) {
  const uint32_t u = __float_as_uint(f + 0.0f);   // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float unord_key(uint32_t k) {
  const uint32_t u = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
  return __uint_as_float(u);
}

struct SelShared {
  uint32_t hist[256];
  uint32_t warp_tot[kSelThreads / 32];
  unsigned long long red[2][kSelThreads / 32][2];
  uint32_t prefix, need, cnt, maxkey, taken_tot;
};

// top-2 of two top-2 lists (keys unique except zeros)
__device__ __forceinline__ void top2_merge(unsigned long long& b1, unsigned long long& b2,
                                           unsigned long long o1, unsigned long long o2) {
  const unsigned long long hi = b1 > o1 ? b1 : o1;
  const unsigned long long lo = b1 > o1 ? o1 : b1;
  const unsigned long long sec = b2 > o2 ? b2 : o2;
  b1 = hi;
  b2 = lo > sec ? lo : sec;
}

// Exclusive prefix count of `flag` over the block in thread order; returns the
// prefix and writes the block total to *total (all threads).
__device__ __forceinline__ uint32_t block_excl_count(bool flag, SelShared& sh, uint32_t* total) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t bal = __ballot_sync(0xffffffffu, flag);
  const uint32_t in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) sh.warp_tot[warp] = __popc(bal);
  __syncthreads();
  uint32_t before = 0, tot = 0;
  for (int w = 0; w < kSelThreads / 32; ++w) {
    const uint32_t x = sh.warp_tot[w];
    if (w < warp) before += x;
    tot += x;
  }
  __syncthreads();
  *total = tot;
  return before + in_warp;
}

__global__ void __launch_bounds__(kSelThreads, 1) select_kernel(const __grid_constant__ SelectParams P) {
  __shared__ SelShared sh;
  extern __shared__ __align__(16) uint8_t dyn[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  const UnitInfo u = unit_info(P.g, blockIdx.x);
  const int W = P.g.window;
  const int Lc = u.L - W;
  const int B = P.budget;
  const int C = P.cand_factor == 0 ? Lc : min(P.cand_factor * B, Lc);
  const int nsel = min(B, C);
  const float lambda1 = P.lambda1[u.layer];
  const float lambda2 = P.lambda2[u.layer];
  const float* mu = P.mu + u.mu_off;
  const float* sg = P.sigma + u.mu_off;
  uint32_t* keys = P.keys + u.mu_off;
  const int h = P.pool_kernel / 2;

  // shared arrays sized by the largest pool
  uint4* kch = reinterpret_cast<uint4*>(dyn);                         // [kChunks][C]
  int32_t* spos = reinterpret_cast<int32_t*>(kch + kChunks * kMaxCand); // [C] sorted positions
  int32_t* cpos = spos + kMaxCand;                                     // [C] collected positions
  float* st = reinterpret_cast<float*>(cpos + kMaxCand);               // [C] s~
  float* inv = st + kMaxCand;                                          // [C] 1/|k|

  // 1. pooled base score as ordered keys
  for (int i = tid; i < Lc; i += kSelThreads) {
    const int lo = max(0, i - h), hi = min(Lc - 1, i + h);
    float mh = mu[lo], sh_ = sg[lo];
    for (int j = lo + 1; j <= hi; ++j) {
      mh = fmaxf(mh, mu[j]);
      sh_ = fmaxf(sh_, sg[j]);
    }
    keys[i] = ord_key(fmaf(lambda1, sh_, mh));
  }
  if (tid == 0) {
    sh.prefix = 0;
    sh.need = static_cast<uint32_t>(C);
    sh.cnt = 0;
    sh.maxkey = 0;
  }
  __syncthreads();

  // 2. radix select of the C-th largest key
  uint32_t pmask = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    if (tid < 256) sh.hist[tid] = 0;
    __syncthreads();
    const uint32_t prefix = sh.prefix;
    for (int i = tid; i < Lc; i += kSelThreads) {
      const uint32_t k = __ldcg(&keys[i]);
      if ((k & pmask) == prefix) atomicAdd(&sh.hist[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      // lane l owns bins 8l .. 8l+7; find the digit where the count from the top
      // first reaches `need`
      uint32_t c[8], s = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) { c[b] = sh.hist[8 * lane + b]; s += c[b]; }
      // inclusive suffix sum over lanes >= lane, then exclusive (lanes > lane)
      uint32_t incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t x = __shfl_down_sync(0xffffffffu, incl, o);
        if (lane + o < 32) incl += x;
      }
      const uint32_t suffix = incl - s;
      const uint32_t need = sh.need;
      int found = -1;
      uint32_t acc = suffix, above_digit = 0;
      if (suffix < need && suffix + s >= need) {
        for (int b = 7; b >= 0; --b) {
          if (acc + c[b] >= need) { found = 8 * lane + b; above_digit = acc; break; }
          acc += c[b];
        }
      }
      const uint32_t bal = __ballot_sync(0xffffffffu, found >= 0);
      const int src = __ffs(bal) - 1;
      const int digit = __shfl_sync(0xffffffffu, found, src);
      const uint32_t abv = __shfl_sync(0xffffffffu, above_digit, src);
      if (lane == 0) {
        sh.prefix = prefix | (static_cast<uint32_t>(digit) << shift);
        sh.need = need - abv;
      }
    }
    pmask |= 0xFFu << shift;
    __syncthreads();
  }
  const uint32_t T = sh.prefix;
  const uint32_t needT = sh.need;   // keys equal to T to take, lowest positions first

  // 3a. every key above the threshold
  for (int i = tid; i < Lc; i += kSelThreads) {
    const uint32_t k = __ldcg(&keys[i]);
    if (k > T) cpos[atomicAdd(&sh.cnt, 1u)] = i;
  }
  __syncthreads();
  const uint32_t n_above = sh.cnt;
  // 3b. the needT lowest positions whose key equals T
  uint32_t taken = 0;
  for (int base = 0; base < Lc && taken < needT; base += kSelThreads) {
    const int i = base + tid;
    const bool f = (i < Lc) && (__ldcg(&keys[i]) == T);
    uint32_t tot;
    const uint32_t pre = block_excl_count(f, sh, &tot);
    if (f && taken + pre < needT) cpos[n_above + taken + pre] = i;
    taken += tot;
  }
  __syncthreads();

  // 4. sort the pool by position, normalise, stage keys and inverse norms
  if (tid < C) {
    const int pos = cpos[tid];
    int rank = 0;
    for (int c = 0; c < C; ++c) rank += (cpos[c] < pos);
    spos[rank] = pos;
    atomicMax(&sh.maxkey, __ldcg(&keys[pos]));
  }
  __syncthreads();
  const float smax = fmaxf(unord_key(sh.maxkey), P.norm_eps);
  float corr = 0.f;
  bool mine_taken = tid >= C;
  if (tid < C) {
    const int pos = spos[tid];
    st[tid] = __fdiv_rn(unord_key(__ldcg(&keys[pos])), smax);
    const uint4* row = reinterpret_cast<const uint4*>(P.k + (u.k_row0 + pos) * kHeadDim);
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < kChunks; ++j) {
      const uint4 x = __ldg(row + j);
      kch[j * kMaxCand + tid] = x;
      const uint32_t w4[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float lo = __uint_as_float(w4[e] << 16);
        const float hi = __uint_as_float(w4[e] & 0xFFFF0000u);
        ss = fmaf(lo, lo, ss);
        ss = fmaf(hi, hi, ss);
      }
    }
    inv[tid] = ss > 0.f ? __fdiv_rn(1.0f, sqrtf(ss)) : 0.f;
  }
  __syncthreads();

  // 5. greedy admissions
  const float my_st = tid < C ? st[tid] : 0.f;
  const float my_inv = tid < C ? inv[tid] : 0.f;
  int32_t* order = P.order ? P.order + u.unit * B : nullptr;
  float* margins = P.margins ? P.margins + u.unit * B : nullptr;
  for (int t = 0; t < nsel; ++t) {
    unsigned long long b1 = 0, b2 = 0;
    if (!mine_taken) {
      const float v = fmaf(lambda2, corr, my_st);
      b1 = (static_cast<unsigned long long>(ord_key(v)) << 32) |
           static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(tid));
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      const unsigned long long o1 = __shfl_xor_sync(0xffffffffu, b1, o);
      const unsigned long long o2 = __shfl_xor_sync(0xffffffffu, b2, o);
      top2_merge(b1, b2, o1, o2);
    }
    if (lane == 0) {
      sh.red[t & 1][warp][0] = b1;
      sh.red[t & 1][warp][1] = b2;
    }
    __syncthreads();
    unsigned long long f1 = 0, f2 = 0;
#pragma unroll
    for (int w = 0; w < kSelThreads / 32; ++w) top2_merge(f1, f2, sh.red[t & 1][w][0], sh.red[t & 1][w][1]);
    const int js = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(f1 & 0xFFFFFFFFull));
    if (tid == 0) {
      if (order) order[t] = spos[js];
      if (margins) {
        const float vb = unord_key(static_cast<uint32_t>(f1 >> 32));
        margins[t] = f2 ? vb - unord_key(static_cast<uint32_t>(f2 >> 32)) : INFINITY;
      }
    }
    if (tid == js) mine_taken = true;
    if (!mine_taken) {
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < kChunks; ++j) {
        const uint4 a = kch[j * kMaxCand + tid];
        const uint4 b = kch[j * kMaxCand + js];
        const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
        const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          dot = fmaf(__uint_as_float(aw[e] << 16), __uint_as_float(bw[e] << 16), dot);
          dot = fmaf(__uint_as_float(aw[e] & 0xFFFF0000u), __uint_as_float(bw[e] & 0xFFFF0000u), dot);
        }
      }
      corr = fmaxf(corr, dot * my_inv * inv[js]);
    }
  }

  // 6. admitted positions in ascending order, then -1
  const bool sel = tid < C && mine_taken;
  uint32_t tot;
  const uint32_t rank = block_excl_count(sel, sh, &tot);
  int32_t* out = P.indices + u.unit * B;
  if (sel) out[rank] = spos[tid];
  for (int r = nsel + tid; r < B; r += kSelThreads) out[r] = -1;
  if (order)
    for (int r = nsel + tid; r < B; r += kSelThreads) order[r] = -1;
  if (margins)
    for (int r = nsel + tid; r < B; r += kSelThreads) margins[r] = 0.f;
}

}  // namespace

cudaError_t launch_select(const kve_plan& plan, const SelectParams& p, cudaStream_t stream) {
  const size_t dyn = kChunks * kMaxCand * sizeof(uint4) + 4 * kMaxCand * sizeof(int32_t);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(dyn));
  if (e != cudaSuccess) return e;
  select_kernel<<<static_cast<unsigned>(plan.geo.n_units), kSelThreads, dyn, stream>>>(p);
  return cudaGetLastError();
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

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
uint32_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_select_scratch on the current device (looked up once per
// device; in host code the symbol itself is only a host-side stand-in).
uint32_t* scratch_on_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_scratch) != cudaSuccess) return nullptr;
    g_scratch_ptr[dev] = static_cast<uint32_t*>(p);
  }
  return g_scratch_ptr[dev];
}

}  // namespace
}  // namespace kve

extern "C" kve_status kv_evict_select_noalloc(const kve_plan* plan, const float* mu, const float* sigma,
                                              const uint16_t* k, const float* lambda1,
                                              const float* lambda2, int32_t* indices, int32_t* order,
                                              float* margins, void* stream) {
  using namespace kve;
  if (!plan || !mu || !sigma || !k || !lambda1 || !lambda2 || !indices) return KVE_EINVAL;
  const Geometry& g = plan->geo;
  const size_t words = static_cast<size_t>(g.num_layers) * g.hkv * static_cast<size_t>(g.total_tokens);
  if (words > kNoAllocScratchWords) return KVE_EINVAL;   // beyond the fixed scratch
  if ((reinterpret_cast<uintptr_t>(k) & 15u) != 0) return KVE_EINVAL;
  uint32_t* scratch = scratch_on_current_device();
  if (!scratch) return KVE_ECUDA;
  SelectParams p;
  memset(&p, 0, sizeof(p));
  p.g = g;
  p.budget = plan->cfg.budget;
  p.pool_kernel = plan->cfg.pool_kernel;
  p.cand_factor = plan->cfg.candidate_factor;
  p.norm_eps = plan->cfg.norm_eps;
  for (int l = 0; l < g.num_layers; ++l) {
    if (!isfinite(lambda1[l]) || !isfinite(lambda2[l])) return KVE_EINVAL;
    p.lambda1[l] = lambda1[l];
    p.lambda2[l] = lambda2[l];
  }
  p.mu = mu;
  p.sigma = sigma;
  p.k = k;
  p.indices = indices;
  p.order = order;
  p.margins = margins;
  p.keys = scratch;
  return launch_select(*plan, p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? KVE_OK : KVE_ECUDA;
}
