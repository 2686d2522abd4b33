// Gather kernel: step 4 of the eviction step (Section 1: after prefill each layer
// keeps B cached entries; the W window tokens are kept as well).
//
// Unit u's compact cache is [B + W][d]: rows 0 .. m-1 are the kept candidates in
// ascending position (m = min(B_l, Lc), B_l the unit's layer budget), rows
// m .. m+W-1 the window tokens Lc .. L-1, the rest zero. A row is 256 bytes, copied by 16 lanes with 16-byte
// accesses, key and value alike; the copy is bit-exact.
#include "kve_internal.h"

namespace kve {
namespace {

constexpr int kGatherThreads = 256;
constexpr int kRowsInFlight = kGatherThreads / 16;   // rows per pass (16 lanes per row)
constexpr int kPasses = 8;                            // passes whose loads are issued together

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const __grid_constant__ GatherParams P) {
  wait_previous_kernel();   // the indices come from the selection launched before
  const UnitInfo u = unit_info(P.g, blockIdx.x);
  const int W = P.g.window;
  const int B = P.budget;
  const int Lc = u.L - W;
  const int m = min(P.layer_budget[u.layer], Lc);
  const int rows = B + W;
  const int half = threadIdx.x >> 4;
  const int lane16 = threadIdx.x & 15;
  const int32_t* idx = P.indices + u.unit * B;
  const uint16_t* ksrc = P.k + u.k_off;           // key i at ksrc + i * k_st (a 16-byte multiple)
  const uint16_t* vsrc = P.v + u.v_off;
  uint4* kdst = reinterpret_cast<uint4*>(P.k_out + u.unit * rows * kHeadDim);
  uint4* vdst = reinterpret_cast<uint4*>(P.v_out + u.unit * rows * kHeadDim);
  // kPasses rows per thread at a time: every load of a batch is in flight before the
  // first store (the rows come from HBM, or from pinned host memory, in place)
  for (int r0 = 0; r0 < rows; r0 += kPasses * kRowsInFlight) {
    int src[kPasses];
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
      const int r = r0 + p * kRowsInFlight + half;
      int s = -1;
      if (r < m) {
        s = __ldg(idx + r);
        if (s < 0 || s >= Lc) s = -1;            // never read outside the unit
      } else if (r < m + W) {
        s = Lc + (r - m);
      }
      src[p] = s;
    }
    uint4 kv[kPasses], vv[kPasses];
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
      kv[p] = make_uint4(0, 0, 0, 0);
      vv[p] = make_uint4(0, 0, 0, 0);
      if (src[p] >= 0) {
        kv[p] = __ldcs(reinterpret_cast<const uint4*>(ksrc + src[p] * P.g.k_st) + lane16);
        vv[p] = __ldcs(reinterpret_cast<const uint4*>(vsrc + src[p] * P.g.v_st) + lane16);
      }
    }
#pragma unroll
    for (int p = 0; p < kPasses; ++p) {
      const int r = r0 + p * kRowsInFlight + half;
      if (r < rows) {
        kdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = kv[p];
        vdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = vv[p];
      }
    }
  }
}

}  // namespace

cudaError_t launch_gather(const kve_plan& plan, const GatherParams& p, cudaStream_t stream) {
  return launch_after_previous(gather_kernel, dim3(static_cast<unsigned>(plan.geo.n_units)),
                               dim3(kGatherThreads), 0, stream, p);
}

}  // namespace kve
