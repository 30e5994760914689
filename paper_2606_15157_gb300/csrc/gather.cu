// gather.cu -- gather-compaction of the kept K/V rows of every SnapKV and H2O
// layer into the packed output cache, in one grid-stride launch (the
// StreamingLLM layers' rows, whose positions need no scores, are copied by the
// selection launch).
//
// Output row (layer l, unit (s, h), slot j) = K[l][s][h][out_idx[row]] and the
// same for V; slots past the kept count (out_idx = -1) are zero-filled.  For
// H2O layers the kept tokens' window scores are gathered too: they seed the
// accumulated-attention state of the decode phase.
//
// Each row is moved as d/8 16-byte vectors (one per thread); a warp covers
// 4 rows (d = 128) or 8 rows (d = 64), so both the loads of one row and the
// stores of consecutive rows are fully coalesced.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

constexpr int kGatherThreads = 256;

// Layer owning gathered row `g`: the last layer whose first gathered row is
// <= g.  FULL and StreamingLLM layers own no gathered rows and share their
// grow_off with the next layer, so the search (which takes the highest such
// index) never lands on them.
__device__ __forceinline__ int find_layer(const GatherParams& p, long long g) {
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.grow_off[mid] <= g) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const __grid_constant__ GatherParams p) {
  const int tpr = p.d / 8;  // threads per row, 16 bytes each
  const int rows_per_block = kGatherThreads / tpr;
  const int sub = threadIdx.x % tpr;
  const long long step = static_cast<long long>(gridDim.x) * rows_per_block;
  for (long long g = static_cast<long long>(blockIdx.x) * rows_per_block + threadIdx.x / tpr;
       g < p.total_rows; g += step) {
    const int l = find_layer(p, g);
    const LayerDesc& ld = p.layer[l];
    const long long local = g - p.grow_off[l];
    const long long row = ld.row_off + local;  // packed output row
    const int rem = static_cast<int>(local / ld.slots);
    int pos = p.out_idx[row];
    if (pos >= p.S_cap) {  // never produced by the selection; guard the loads anyway
      if (sub == 0) atomicOr(p.status, kStatusDevice);
      pos = -1;
    }
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (pos >= 0) {
      const size_t src = (static_cast<size_t>(rem) * p.S_cap + pos) * p.d + sub * 8;
      kv = __ldg(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p.K[l]) + src));
      vv = __ldg(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(p.V[l]) + src));
    }
    const size_t dst = static_cast<size_t>(row) * p.d + sub * 8;
    __stcs(reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.out_K) + dst), kv);
    __stcs(reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.out_V) + dst), vv);
    if (sub == 0 && ld.method == KVEV_H2O && p.h2o_state != nullptr) {
      float a = 0.f;
      if (pos >= 0)
        a = ld.scores[static_cast<size_t>(rem) * p.S_cap + pos];
      p.h2o_state[row] = a;
    }
  }
}

}  // namespace

cudaError_t launch_gather(const GatherParams& p, cudaStream_t s, int num_sms) {
  if (p.total_rows == 0) return cudaSuccess;
  const int rows_per_block = kGatherThreads / (p.d / 8);
  long long blocks = (p.total_rows + rows_per_block - 1) / rows_per_block;
  const long long cap = static_cast<long long>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  gather_kernel<<<static_cast<int>(blocks), kGatherThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
