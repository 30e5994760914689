// select.cu -- per (layer, sequence, KV head) choice of the positions to keep,
// for every non-FULL layer of the route in one launch (one CTA per unit).
//
//   SnapKV   : E = n - W prefix positions; keys = 1-D pooled window scores
//              (stride 1, width p, same length; max ignores out-of-range
//              entries, avg pads with zeros and divides by p); keep the
//              top (b - W) prefix positions plus the window [E, n).
//   H2O      : E = n - r (r = protected recent window); keys = raw window
//              scores; keep the top (b - r) of [0, E) plus [E, n).
//   Streaming: keep [0, sink) plus the last `recent` positions (closed form).
//   b >= n   : keep every position.
// Top-k order: larger score first, equal scores keep the lower position.
// Output indices are ascending; unused slots hold -1.
//
// The k-th largest key is found by a 4-pass 8-bit radix select over an
// order-preserving uint32 image of the fp32 scores held in shared memory,
// then one ordered pass (ballot/popc prefix counts) writes the kept positions.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

// Per-unit scores (or pooled scores) into order-preserving keys in shared
// memory.  Every load of a key's window is issued before any is used, four
// keys per thread at a time (the window reads of neighbouring keys overlap
// and are served by L1), so the latency of the score reads is paid once per
// group of keys rather than once per window element.
template <int P>
__device__ __forceinline__ void build_keys_pooled(uint32_t* keys, const float* raw, int E, bool is_max) {
  constexpr int h = P / 2;
  constexpr int U = 4;
  for (int i0 = threadIdx.x; i0 < E; i0 += U * blockDim.x) {
    float w[U][P];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i0 + u * blockDim.x;
#pragma unroll
      for (int j = 0; j < P; ++j) {
        const int q = i - h + j;
        w[u][j] = (i < E && q >= 0 && q < E) ? raw[q] : (is_max ? -INFINITY : 0.f);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = i0 + u * blockDim.x;
      if (i >= E) break;
      float v = w[u][0];
#pragma unroll
      for (int j = 1; j < P; ++j) v = is_max ? fmaxf(v, w[u][j]) : v + w[u][j];
      keys[i] = float_key(is_max ? v : v / static_cast<float>(P));
    }
  }
}

__device__ void build_keys(uint32_t* keys, const float* raw, int E, int pool, int pool_type,
                           bool do_pool) {
  const bool is_max = pool_type == KVEV_POOL_MAX;
  if (do_pool) {
    switch (pool) {  // common widths with fully unrolled windows
      case 3: build_keys_pooled<3>(keys, raw, E, is_max); return;
      case 5: build_keys_pooled<5>(keys, raw, E, is_max); return;
      case 7: build_keys_pooled<7>(keys, raw, E, is_max); return;
      case 9: build_keys_pooled<9>(keys, raw, E, is_max); return;
      default: break;
    }
  }
  const int h = pool / 2;
  for (int i = threadIdx.x; i < E; i += blockDim.x) {
    float v;
    if (!do_pool) {
      v = raw[i];
    } else if (is_max) {
      v = -INFINITY;
      const int lo = max(i - h, 0), hi = min(i + h, E - 1);
      for (int j = lo; j <= hi; ++j) v = fmaxf(v, raw[j]);
    } else {
      float sum = 0.f;
      const int lo = max(i - h, 0), hi = min(i + h, E - 1);
      for (int j = lo; j <= hi; ++j) sum += raw[j];
      v = sum / static_cast<float>(pool);
    }
    keys[i] = float_key(v);
  }
}

struct SelShared {
  int hist[256];
  int wcnt[2][32];
  int bcast[4];
};

// Threshold key T (the k-th largest) and how many keys equal to T to keep.
__device__ void radix_select(const uint32_t* keys, int E, int k, SelShared& sh, uint32_t& T,
                             int& need) {
  uint32_t prefix = 0, mask = 0;
  int kk = k;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) sh.hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < E; base += blockDim.x) {
      const int i = base + threadIdx.x;
      const bool in = i < E && (keys[i] & mask) == prefix;
      const uint32_t digit = in ? (keys[i] >> shift) & 255u : 256u;
      const uint32_t peers = __match_any_sync(0xffffffffu, digit);
      if (in && lane == __ffs(peers) - 1) atomicAdd(&sh.hist[digit], __popc(peers));
    }
    __syncthreads();
    if (warp == 0) {
      // bins in descending digit order; lane l owns digits 255-8l ... 248-8l
      int c[8], s = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        c[q] = sh.hist[255 - 8 * lane - q];
        s += c[q];
      }
      int incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int before = incl - s;
      if (before < kk && kk <= incl) {
        int acc = before, q = 0;
        while (acc + c[q] < kk) acc += c[q++];
        sh.bcast[0] = 255 - 8 * lane - q;  // selected digit
        sh.bcast[1] = acc;                 // keys with a larger digit (within prefix)
      }
    }
    __syncthreads();
    const uint32_t dsel = static_cast<uint32_t>(sh.bcast[0]);
    kk -= sh.bcast[1];
    prefix |= dsel << shift;
    mask |= 255u << shift;
    __syncthreads();
  }
  T = prefix;
  need = kk;
}

// Ordered write of the selected positions of [0, E) to out[0..k).
__device__ void compact(const uint32_t* keys, int E, int k, uint32_t T, int need, SelShared& sh,
                        int* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = blockDim.x >> 5;
  const int seg = (((E + nwarps - 1) / nwarps) + 31) & ~31;
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int gt = 0, eq = 0;
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int i = b0 + lane;
    const uint32_t key = i < hi ? keys[i] : 0u;
    gt += __popc(__ballot_sync(0xffffffffu, i < hi && key > T));
    eq += __popc(__ballot_sync(0xffffffffu, i < hi && key == T));
  }
  if (lane == 0) {
    sh.wcnt[0][warp] = gt;
    sh.wcnt[1][warp] = eq;
  }
  __syncthreads();
  int eq_base = 0, sel_base = 0;
  for (int w = 0; w < warp; ++w) {
    const int e = sh.wcnt[1][w];
    const int take = min(max(need - eq_base, 0), e);
    sel_base += sh.wcnt[0][w] + take;
    eq_base += e;
  }
  const uint32_t lt = (1u << lane) - 1u;
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int i = b0 + lane;
    const uint32_t key = i < hi ? keys[i] : 0u;
    const bool g = i < hi && key > T;
    const bool e = i < hi && key == T;
    const uint32_t eb = __ballot_sync(0xffffffffu, e);
    const int rank = eq_base + __popc(eb & lt);
    const bool sel = g || (e && rank < need);
    const uint32_t sb = __ballot_sync(0xffffffffu, sel);
    const int slot = sel_base + __popc(sb & lt);
    if (sel && slot < k) out[slot] = i;
    eq_base += __popc(eb);
    sel_base += __popc(sb);
  }
}

__global__ void __launch_bounds__(kSelectThreads) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ uint32_t keys[];
  __shared__ SelShared sh;
  const int per_layer = p.B * p.H_kv;
  const int l = blockIdx.x / per_layer;
  const int rem = blockIdx.x - l * per_layer;
  const int s = rem / p.H_kv;
  const LayerDesc ld = p.layer[l];
  const int n = p.lens[s];
  int* cnt = p.out_count + static_cast<size_t>(l) * per_layer + rem;
  if (ld.method == KVEV_FULL) {
    if (threadIdx.x == 0) *cnt = n;
    return;
  }
  const int b = ld.slots;
  int* idx = p.out_idx + ld.row_off + static_cast<long long>(rem) * b;

  int count, E = n, k = 0;  // select top-k of [0, E), then keep [E, n)
  bool identity = false;
  if (ld.method == KVEV_STREAMING) {
    const int cap = p.sink + ld.recent;
    identity = n <= cap;
    count = identity ? n : cap;
    if (!identity) {
      for (int j = threadIdx.x; j < count; j += blockDim.x)
        idx[j] = j < p.sink ? j : n - ld.recent + (j - p.sink);
    }
  } else {
    identity = n <= b;
    count = identity ? n : b;
    if (!identity) {
      const int protect = ld.method == KVEV_SNAPKV ? p.W : ld.h2o_recent;
      E = n - protect;
      k = b - protect;
    }
  }
  if (identity)
    for (int j = threadIdx.x; j < n; j += blockDim.x) idx[j] = j;
  for (int j = count + threadIdx.x; j < b; j += blockDim.x) idx[j] = -1;
  if (threadIdx.x == 0) *cnt = count;
  if (identity || ld.method == KVEV_STREAMING) return;

  // protected tail [E, n) occupies slots k .. count-1
  for (int j = threadIdx.x; j < n - E; j += blockDim.x) idx[k + j] = E + j;
  if (k == 0) return;
  const float* raw =
      p.raw + (static_cast<size_t>(ld.score_slot) * per_layer + rem) * static_cast<size_t>(p.S_cap);
  build_keys(keys, raw, E, p.pool_kernel, p.pool_type, ld.method == KVEV_SNAPKV);
  __syncthreads();
  if (k >= E) {
    for (int j = threadIdx.x; j < E; j += blockDim.x) idx[j] = j;
    return;
  }
  uint32_t T;
  int need;
  radix_select(keys, E, k, sh, T, need);
  compact(keys, E, k, T, need, sh, idx);
}

}  // namespace

cudaError_t select_set_smem(size_t smem) {
  return cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

cudaError_t launch_select(const SelectParams& p, int grid, size_t smem, cudaStream_t s) {
  if (grid == 0) return cudaSuccess;
  select_kernel<<<grid, kSelectThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
