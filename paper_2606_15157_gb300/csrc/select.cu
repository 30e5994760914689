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
// The k-th largest key is found over an order-preserving uint32 image of the
// fp32 scores held in shared memory.  The pass that builds the keys also
// histograms their top 12 bits; the bin holding the k-th key is then the only
// one that matters: each warp counts, then gathers in position order, that
// bin's positions in its segment (counting the keys above it), two 10-bit
// radix passes over those candidates alone fix the threshold key, and one
// ordered pass (ballot/popc prefix counts) writes the kept positions.  Four
// light passes over the unit's keys in all, none through a shared counter; a
// first bin too crowded for the candidate buffer takes four 8-bit radix
// passes over every key instead.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

// Bulk prefetch of [src, src + bytes) into L2 (src 16-byte aligned, bytes a
// multiple of 16).
__device__ __forceinline__ void prefetch_l2_bulk(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

constexpr int kHistBits = 12;              // first radix digit: the top 12 bits of a key
constexpr int kHistBins = 1 << kHistBits;
constexpr int kSelWarps = kSelectThreads / 32;

static_assert(kSelWarps == 32, "find_bin scans the warp totals with one warp");

struct SelShared {
  int hist[kHistBins];
  int wsum[kSelWarps];
  int wcnt[2][kSelWarps];  // per warp segment: keys above T, keys equal to T
  int bcast[2];
  int ncand;
};

// Adds each valid lane's digit to the histogram, one shared-memory atomic per
// distinct digit of the warp (the scores of a unit crowd into few bins).
// Every lane of the warp must call it.
__device__ __forceinline__ void hist_add(int* hist, bool valid, uint32_t digit) {
  const uint32_t d = valid ? digit : 0xFFFFFFFFu;
  const uint32_t peers = __match_any_sync(0xffffffffu, d);
  if (valid && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[d], __popc(peers));
}

// Per-unit scores (or pooled scores) into order-preserving keys in shared
// memory, and the histogram of their top kHistBits bits.  Every load of a
// key's window is issued before any is used, four keys per thread at a time
// (the window reads of neighbouring keys overlap and are served by L1), so the
// latency of the score reads is paid once per group of keys rather than once
// per window element.  The loop bounds are uniform over the block so that all
// lanes reach the warp-wide match in hist_add.
template <int P>
__device__ __forceinline__ void build_keys_pooled(uint32_t* keys, int* hist, const float* raw, int E,
                                                  bool is_max) {
  constexpr int h = P / 2;
  constexpr int U = 4;
  for (int b0 = 0; b0 < E; b0 += U * kSelectThreads) {
    float w[U][P];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = b0 + u * kSelectThreads + threadIdx.x;
#pragma unroll
      for (int j = 0; j < P; ++j) {
        const int q = i - h + j;
        w[u][j] = (i < E && q >= 0 && q < E) ? raw[q] : (is_max ? -INFINITY : 0.f);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int i = b0 + u * kSelectThreads + threadIdx.x;
      float v = w[u][0];
#pragma unroll
      for (int j = 1; j < P; ++j) v = is_max ? fmaxf(v, w[u][j]) : v + w[u][j];
      const uint32_t key = float_key(is_max ? v : v / static_cast<float>(P));
      if (i < E) keys[i] = key;
      hist_add(hist, i < E, key >> (32 - kHistBits));
    }
  }
}

// The same with 16-byte loads, for a 16-byte aligned score row: thread t of a
// round takes keys 4t .. 4t+3, whose windows (P <= 9) lie in the three
// aligned 4-float chunks starting at 4t - 4, 4t and 4t + 4.  Only chunks that
// start before E are read (E <= S_cap, a multiple of 4, so none leaves the
// row); entries outside [0, E) count as -inf (max) or 0 (avg).
template <int P>
__device__ __forceinline__ void build_keys_pooled4(uint32_t* keys, int* hist, const float* raw, int E,
                                                   bool is_max) {
  constexpr int h = P / 2;
  static_assert(h <= 4, "the three chunks cover windows of up to 9");
  const float fill = is_max ? -INFINITY : 0.f;
  for (int b0 = 0; b0 < E; b0 += 4 * kSelectThreads) {
    const int i0 = b0 + 4 * threadIdx.x;  // first of this thread's four keys
    float w[12];
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const int st = i0 - 4 + 4 * c;
      float4 v = make_float4(fill, fill, fill, fill);
      if (st >= 0 && st < E) v = *reinterpret_cast<const float4*>(raw + st);
      w[4 * c + 0] = st + 0 < E ? v.x : fill;
      w[4 * c + 1] = st + 1 < E ? v.y : fill;
      w[4 * c + 2] = st + 2 < E ? v.z : fill;
      w[4 * c + 3] = st + 3 < E ? v.w : fill;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u;
      float v = w[4 + u - h];
#pragma unroll
      for (int j = 1; j < P; ++j) v = is_max ? fmaxf(v, w[4 + u - h + j]) : v + w[4 + u - h + j];
      const uint32_t key = float_key(is_max ? v : v / static_cast<float>(P));
      if (i < E) keys[i] = key;
      hist_add(hist, i < E, key >> (32 - kHistBits));
    }
  }
}

__device__ void build_keys(uint32_t* keys, int* hist, const float* raw, int E, int pool, int pool_type,
                           bool do_pool, bool aligned4) {
  const bool is_max = pool_type == KVEV_POOL_MAX;
  if (do_pool && aligned4) {
    switch (pool) {
      case 3: build_keys_pooled4<3>(keys, hist, raw, E, is_max); return;
      case 5: build_keys_pooled4<5>(keys, hist, raw, E, is_max); return;
      case 7: build_keys_pooled4<7>(keys, hist, raw, E, is_max); return;
      case 9: build_keys_pooled4<9>(keys, hist, raw, E, is_max); return;
      default: break;
    }
  }
  if (do_pool) {
    switch (pool) {  // common widths with fully unrolled windows
      case 3: build_keys_pooled<3>(keys, hist, raw, E, is_max); return;
      case 5: build_keys_pooled<5>(keys, hist, raw, E, is_max); return;
      case 7: build_keys_pooled<7>(keys, hist, raw, E, is_max); return;
      case 9: build_keys_pooled<9>(keys, hist, raw, E, is_max); return;
      default: break;
    }
  }
  const int h = pool / 2;
  for (int b0 = 0; b0 < E; b0 += kSelectThreads) {
    const int i = b0 + threadIdx.x;
    float v = 0.f;
    if (i < E) {
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
    }
    const uint32_t key = float_key(v);
    if (i < E) keys[i] = key;
    hist_add(hist, i < E, key >> (32 - kHistBits));
  }
}

// The bin of a histogram of `nbins` digits (a multiple of the block size)
// that holds the kk-th largest key (kk >= 1), and the number of keys in
// higher bins.  Thread t owns bins nbins-1-q*t .. nbins-q*t-q (descending).
__device__ void find_bin(SelShared& sh, int nbins, int kk, int& digit, int& above) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q = nbins / kSelectThreads;
  const int top = nbins - 1 - q * threadIdx.x;
  int s = 0;
  for (int j = 0; j < q; ++j) s += sh.hist[top - j];
  int incl = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) sh.wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = sh.wsum[lane], wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += y;
    }
    sh.wsum[lane] = wi - w;  // exclusive prefix over warps
  }
  __syncthreads();
  incl += sh.wsum[warp];
  const int before = incl - s;
  if (before < kk && kk <= incl) {
    int acc = before, j = 0;
    while (j < q - 1 && acc + sh.hist[top - j] < kk) acc += sh.hist[top - j++];
    sh.bcast[0] = top - j;
    sh.bcast[1] = acc;
  }
  __syncthreads();
  digit = sh.bcast[0];
  above = sh.bcast[1];
  __syncthreads();
}

// Threshold key T (the k-th largest) and how many keys equal to T to keep,
// by 8-bit radix passes over every key (the general path).
__device__ void radix_select(const uint32_t* keys, int E, int k, SelShared& sh, uint32_t& T,
                             int& need) {
  uint32_t prefix = 0, mask = 0;
  int kk = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < kHistBins; i += kSelectThreads) sh.hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < E; base += kSelectThreads) {
      const int i = base + threadIdx.x;
      const bool in = i < E && (keys[i] & mask) == prefix;
      hist_add(sh.hist, in, in ? (keys[i] >> shift) & 255u : 0u);
    }
    __syncthreads();
    int digit, above;  // bins 256 .. 1023 are empty: the 1024-bin search ends in 255 .. 0

    find_bin(sh, 1024, kk, digit, above);
    kk -= above;
    prefix |= static_cast<uint32_t>(digit) << shift;
    mask |= 255u << shift;
  }
  T = prefix;
  need = kk;
}

// Warp segments of [0, E): contiguous, 32-aligned, in warp order, so that a
// warp's kept positions follow those of the warps before it.
__device__ __forceinline__ int seg_len(int E) { return (((E + kSelWarps - 1) / kSelWarps) + 31) & ~31; }

// Ordered write of the kept positions of [0, E) to out[0..k): keys above T,
// and the first `need` keys equal to T in position order.  sh.wcnt holds each
// warp segment's counts of both.
__device__ void write_kept(const uint32_t* keys, int E, int k, uint32_t T, int need, SelShared& sh,
                           int* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
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

// Per-warp-segment counts of keys above and equal to T over all of [0, E).
__device__ void count_segments(const uint32_t* keys, int E, uint32_t T, SelShared& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
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
}

// The fast path once the first digit's bin (digit d0, kk-th within it) holds
// at most `cap` keys.  Each warp counts its segment's keys of that bin and of
// higher bins; a block prefix over the warps gives each warp its own range of
// cand[], which it fills in position order (no shared counter).  The remaining
// 20 bits are resolved by two 10-bit radix passes over the candidates alone
// (their digits are spread out, so plain shared-memory atomics), and each warp
// then counts its own candidates above and equal to T.
__device__ void select_by_candidates(const uint32_t* keys, int E, uint32_t d0, int kk, SelShared& sh,
                                     int* cand, uint32_t& T, int& need) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  const uint32_t lt = (1u << lane) - 1u;
  int gt = 0, mine = 0;
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int i = b0 + lane;
    const uint32_t d = i < hi ? keys[i] >> (32 - kHistBits) : 0u;
    gt += __popc(__ballot_sync(0xffffffffu, i < hi && d > d0));
    mine += __popc(__ballot_sync(0xffffffffu, i < hi && d == d0));
  }
  if (lane == 0) sh.wsum[warp] = mine;
  __syncthreads();
  if (warp == 0) {  // exclusive prefix of the per-warp candidate counts
    const int v = sh.wsum[lane];
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    sh.wsum[lane] = incl - v;
    if (lane == 31) sh.ncand = incl;
  }
  __syncthreads();
  const int first = sh.wsum[warp];  // this warp's range of cand[]: [first, first + mine)
  int at = first;
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int i = b0 + lane;
    const bool in = i < hi && (keys[i] >> (32 - kHistBits)) == d0;
    const uint32_t b = __ballot_sync(0xffffffffu, in);
    if (in) cand[at + __popc(b & lt)] = i;
    at += __popc(b);
  }
  __syncthreads();
  const int nc = sh.ncand;
  uint32_t prefix = d0 << (32 - kHistBits), mask = ~0u << (32 - kHistBits);
  for (int shift = 10; shift >= 0; shift -= 10) {
    for (int i = threadIdx.x; i < 1024; i += kSelectThreads) sh.hist[i] = 0;
    __syncthreads();
    for (int c = threadIdx.x; c < nc; c += kSelectThreads) {
      const uint32_t key = keys[cand[c]];
      if ((key & mask) == prefix) atomicAdd(&sh.hist[(key >> shift) & 1023u], 1);
    }
    __syncthreads();
    int digit, above;
    find_bin(sh, 1024, kk, digit, above);
    kk -= above;
    prefix |= static_cast<uint32_t>(digit) << shift;
    mask |= 1023u << shift;
  }
  T = prefix;
  need = kk;
  int eq = 0;
  for (int c0 = 0; c0 < mine; c0 += 32) {
    const bool v = c0 + lane < mine;
    const uint32_t key = v ? keys[cand[first + c0 + lane]] : 0u;
    gt += __popc(__ballot_sync(0xffffffffu, v && key > T));
    eq += __popc(__ballot_sync(0xffffffffu, v && key == T));
  }
  if (lane == 0) {
    sh.wcnt[0][warp] = gt;
    sh.wcnt[1][warp] = eq;
  }
  __syncthreads();
}

static_assert(sizeof(SelShared) <= kSelectStaticSmem, "select kernel's static shared memory");

template <bool kKeysInWorkspace>
__global__ void __launch_bounds__(kSelectThreads) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ uint32_t keys_smem[];
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
  if (k >= E) {
    for (int j = threadIdx.x; j < E; j += blockDim.x) idx[j] = j;
    return;
  }
  const float* raw = ld.scores + static_cast<size_t>(rem) * p.S_cap;
  // the unit's keys, then its candidate positions: shared memory, or the
  // workspace for capacities whose keys do not fit
  uint32_t* keys = kKeysInWorkspace
                       ? p.keys_g + (static_cast<size_t>(ld.score_slot) * per_layer + rem) * 2 * p.S_cap
                       : keys_smem;
  // pull the unit's scores into L2 in 16 KiB pieces (16-byte aligned, whole
  // 16-byte blocks: the score array is one 256-byte aligned workspace region)
  {
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(raw) & ~uintptr_t(15);
    const uintptr_t a1 = (reinterpret_cast<uintptr_t>(raw + E) + 15) & ~uintptr_t(15);
    const uintptr_t a = a0 + static_cast<uintptr_t>(threadIdx.x) * 16384;
    if (a < a1) prefetch_l2_bulk(reinterpret_cast<const void*>(a), static_cast<uint32_t>(a1 - a < 16384 ? a1 - a : 16384));
  }
  for (int i = threadIdx.x; i < kHistBins; i += kSelectThreads) sh.hist[i] = 0;
  __syncthreads();
  const bool aligned4 = (reinterpret_cast<uintptr_t>(raw) & 15u) == 0 && (p.S_cap & 3) == 0;
  build_keys(keys, sh.hist, raw, E, p.pool_kernel, p.pool_type, ld.method == KVEV_SNAPKV, aligned4);
  __syncthreads();
  int d0, above;
  find_bin(sh, kHistBins, k, d0, above);
  uint32_t T;
  int need;
  if (sh.hist[d0] <= p.cand_cap) {
    select_by_candidates(keys, E, static_cast<uint32_t>(d0), k - above, sh,
                         reinterpret_cast<int*>(keys + p.S_cap), T, need);
  } else {  // a crowded first bin (e.g. many equal scores): radix passes over every key
    radix_select(keys, E, k, sh, T, need);
    count_segments(keys, E, T, sh);
  }
  write_kept(keys, E, k, T, need, sh, idx);
}

}  // namespace

cudaError_t select_set_smem(size_t smem) {
  return cudaFuncSetAttribute(select_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

cudaError_t launch_select(const SelectParams& p, int grid, size_t smem, cudaStream_t s) {
  if (grid == 0) return cudaSuccess;
  if (p.keys_g != nullptr)
    select_kernel<true><<<grid, kSelectThreads, 0, s>>>(p);
  else
    select_kernel<false><<<grid, kSelectThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
