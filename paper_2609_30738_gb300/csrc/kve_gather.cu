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

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const __grid_constant__ GatherParams P) {
  const UnitInfo u = unit_info(P.g, blockIdx.x);
  const int W = P.g.window;
  const int B = P.budget;
  const int Lc = u.L - W;
  const int m = min(P.layer_budget[u.layer], Lc);
  const int rows = B + W;
  const int half = threadIdx.x >> 4;            // 16 rows in flight per block
  const int lane16 = threadIdx.x & 15;
  const int32_t* idx = P.indices + u.unit * B;
  const uint4* ksrc = reinterpret_cast<const uint4*>(P.k + u.k_row0 * kHeadDim);
  const uint4* vsrc = reinterpret_cast<const uint4*>(P.v + u.k_row0 * kHeadDim);
  uint4* kdst = reinterpret_cast<uint4*>(P.k_out + u.unit * rows * kHeadDim);
  uint4* vdst = reinterpret_cast<uint4*>(P.v_out + u.unit * rows * kHeadDim);
  for (int r = half; r < rows; r += kGatherThreads / 16) {
    int src = -1;
    if (r < m) {
      src = __ldg(idx + r);
      if (src < 0 || src >= Lc) src = -1;       // never read outside the unit
    } else if (r < m + W) {
      src = Lc + (r - m);
    }
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (src >= 0) {
      kv = __ldcs(ksrc + static_cast<int64_t>(src) * (kHeadDim / 8) + lane16);
      vv = __ldcs(vsrc + static_cast<int64_t>(src) * (kHeadDim / 8) + lane16);
    }
    kdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = kv;
    vdst[static_cast<int64_t>(r) * (kHeadDim / 8) + lane16] = vv;
  }
}

}  // namespace

cudaError_t launch_gather(const kve_plan& plan, const GatherParams& p, cudaStream_t stream) {
  gather_kernel<<<static_cast<unsigned>(plan.geo.n_units), kGatherThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace kve
