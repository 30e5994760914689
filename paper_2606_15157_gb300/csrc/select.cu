// select.cu -- per (layer, sequence, KV head) choice of the positions to keep,
// for every non-FULL layer of the route in one launch (one CTA per unit).
//
//   SnapKV   : E = n - W prefix positions; keys = 1-D pooled window scores
//              (stride 1, width p, same length; max ignores out-of-range
//              entries, avg pads with zeros and divides by p -- a division
//              by the same p for every key, so the window sum ranks the keys
//              alike and is used instead); keep the top (b - W) prefix
//              positions plus the window [E, n).
//   H2O      : E = n - r (r = protected recent window); keys = raw window
//              scores; keep the top (b - r) of [0, E) plus [E, n).
//   Streaming: keep [0, sink) plus the last `recent` positions (closed form).
//   b >= n   : keep every position.
// Top-k order: larger score first, equal scores keep the lower position.
// Output indices are ascending; unused slots hold -1.
//
// A unit takes a CTA of 256 threads, so that several units share an SM and
// one unit's barriers and round trips overlap another's passes.  The keys (an
// order-preserving uint32 image of the fp32 scores) go to the unit's row of a
// workspace array, which stays in L2 between the passes:
//   1. build the keys and find their range [lo, hi];
//   2. histogram the first digit (key - lo) >> s, which splits the range into
//      at most 8192 bins of 2^s keys (a unit's scores may crowd into a few
//      per cent of one octave, or spread over many octaves: the range adapts
//      the bins to either);
//   3. find the bin holding the k-th largest key; each warp counts the keys
//      of higher bins in its segment and appends that bin's keys (the
//      candidates) to a shared list that reuses the histogram's space; radix
//      passes of up to 9 bits over the candidates' s low bits fix the
//      threshold key T and how many keys equal to T to keep, and the
//      candidates' tallies give every warp segment its counts above and equal
//      to T;
//   4. one ordered pass writes the kept positions: a warp's slots follow those
//      of the warps before it, and within a warp lanes hold four consecutive
//      keys each, ranked by warp scans.
// Equal keys everywhere take the first k positions directly; a candidate bin
// with more keys than the list holds (many equal keys) takes four 8-bit radix
// passes over every key instead.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

constexpr int kSW = kSelectThreads / 32;   // warps of a selection CTA
constexpr int kBins0 = 8192;               // first digit: the keys' range in at most 8192 bins
constexpr int kCandCap = kBins0 / 2;       // (position, key) pairs in the histogram's space
constexpr int kBins1 = 512;                // candidate digits: up to 9 bits a pass
constexpr int kSegKeys = 128;              // a warp block: four keys per lane
constexpr int kSelectUnroll = 4;           // key blocks whose loads are in flight together

struct __align__(16) SelShared {
  union {
    int hist[kBins0];
    uint2 cand[kCandCap];
  } u;
  int hist1[kBins1];
  int wsum[kSW];
  int wgt[kSW];   // per warp segment: keys above T
  int weq[kSW];   // per warp segment: keys equal to T
  int bcast[2];
  int ncand;
};

static_assert(sizeof(SelShared) <= 48 * 1024, "the selection's shared memory is static");

// Adds each valid lane's digit to the histogram, one shared-memory atomic per
// distinct digit of the warp (the scores of a unit crowd into few bins).
// Every lane of the warp must call it.
__device__ __forceinline__ void hist_add(int* hist, bool valid, uint32_t digit) {
  const uint32_t d = valid ? digit : 0xFFFFFFFFu;
  const uint32_t peers = __match_any_sync(0xffffffffu, d);
  if (valid && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[d], __popc(peers));
}

// Inclusive warp scan.
__device__ __forceinline__ int warp_incl(int x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

__device__ __forceinline__ int warp_sum(int x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// The bin of a histogram of `nbins` digits (a multiple of the block size)
// that holds the kk-th largest key (1 <= kk <= keys counted), and the number
// of keys in higher bins.  Thread t owns the q = nbins / 256 bins
// nbins-1-q*t down to nbins-q*(t+1).
__device__ void find_bin(const int* hist, int nbins, int kk, SelShared& sh, int& digit, int& above) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int q = nbins / kSelectThreads;
  const int lo = nbins - q * (threadIdx.x + 1);  // this thread's lowest bin
  int s = 0;
  if (q % 4 == 0) {
    const int4* h4 = reinterpret_cast<const int4*>(hist + lo);
    for (int j = 0; j < q / 4; ++j) {
      const int4 v = h4[j];
      s += (v.x + v.y) + (v.z + v.w);
    }
  } else {
    for (int j = 0; j < q; ++j) s += hist[lo + j];
  }
  int incl = warp_incl(s);
  if (lane == 31) sh.wsum[warp] = incl;
  __syncthreads();
  for (int w = 0; w < warp; ++w) incl += sh.wsum[w];
  const int before = incl - s;
  if (before < kk && kk <= incl) {
    int acc = before, b = lo + q - 1;
    while (b > lo && acc + hist[b] < kk) acc += hist[b--];
    sh.bcast[0] = b;
    sh.bcast[1] = acc;
  }
  __syncthreads();
  digit = sh.bcast[0];
  above = sh.bcast[1];
  __syncthreads();  // wsum and bcast are reused by the next call
}

// Warp segments of [0, E): contiguous, whole 128-key iterations, in warp
// order, so that a warp's kept positions follow those of the warps before it.
__device__ __forceinline__ int seg_len(int E) {
  return ((E + kSW - 1) / kSW + kSegKeys - 1) / kSegKeys * kSegKeys;
}

// Four consecutive keys from a 16-byte aligned key row (the row is padded to
// a multiple of four entries, so the load never leaves it).
__device__ __forceinline__ uint4 ld_keys4(const uint32_t* keys, int i0) {
  return __ldcg(reinterpret_cast<const uint4*>(keys + i0));
}

__device__ __forceinline__ uint32_t pick(const uint4& v, int u) {
  return u == 0 ? v.x : u == 1 ? v.y : u == 2 ? v.z : v.w;
}

// ---------------------------------------------------------------------------
// Pass 1: the keys and their range.  Keys past E in the last group of four are
// written too (the row is padded); no later pass reads them.
// ---------------------------------------------------------------------------
struct KeyRange {
  uint32_t lo = 0xFFFFFFFFu, hi = 0u;
  __device__ __forceinline__ void add(uint32_t k, bool valid) {
    if (valid) {
      lo = min(lo, k);
      hi = max(hi, k);
    }
  }
};

// Pooled keys from a 16-byte aligned score row: thread t of a round takes keys
// 4t .. 4t+3, whose windows (P <= 9) lie in the three aligned 4-float chunks
// starting at 4t - 4, 4t and 4t + 4.  Only chunks that start before E are read
// (E <= S_cap, a multiple of 4, so none leaves the row); entries outside
// [0, E) count as -inf (max) or 0 (avg).
template <int P>
__device__ __forceinline__ void build_pooled4(uint32_t* keys, const float* raw, int E, bool is_max,
                                              KeyRange& kr) {
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
      if (st >= 0 && st < E) v = __ldg(reinterpret_cast<const float4*>(raw + st));  // neighbours' chunks: L1 hits
      w[4 * c + 0] = st + 0 < E ? v.x : fill;
      w[4 * c + 1] = st + 1 < E ? v.y : fill;
      w[4 * c + 2] = st + 2 < E ? v.z : fill;
      w[4 * c + 3] = st + 3 < E ? v.w : fill;
    }
    uint32_t kq[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      float v = w[4 + u - h];
#pragma unroll
      for (int j = 1; j < P; ++j) v = is_max ? fmaxf(v, w[4 + u - h + j]) : v + w[4 + u - h + j];
      kq[u] = float_key(v);
      kr.add(kq[u], i0 + u < E);
    }
    if (i0 < E) *reinterpret_cast<uint4*>(keys + i0) = make_uint4(kq[0], kq[1], kq[2], kq[3]);
  }
}

// Raw keys (no pooling) from a 16-byte aligned score row.
__device__ __forceinline__ void build_raw4(uint32_t* keys, const float* raw, int E, KeyRange& kr) {
  for (int b0 = 0; b0 < E; b0 += 4 * kSelectThreads) {
    const int i0 = b0 + 4 * threadIdx.x;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 < E) v = __ldg(reinterpret_cast<const float4*>(raw + i0));
    const uint32_t kq[4] = {float_key(v.x), float_key(v.y), float_key(v.z), float_key(v.w)};
#pragma unroll
    for (int u = 0; u < 4; ++u) kr.add(kq[u], i0 + u < E);
    if (i0 < E) *reinterpret_cast<uint4*>(keys + i0) = make_uint4(kq[0], kq[1], kq[2], kq[3]);
  }
}

// Any alignment and any odd pooling width: one key per thread at a time.
__device__ void build_scalar(uint32_t* keys, const float* raw, int E, int pool, bool do_pool, bool is_max,
                             KeyRange& kr) {
  const int h = pool / 2;
  for (int i = threadIdx.x; i < E; i += kSelectThreads) {
    float v;
    if (!do_pool) {
      v = raw[i];
    } else if (is_max) {
      v = -INFINITY;
      const int lo = max(i - h, 0), hi = min(i + h, E - 1);
      for (int j = lo; j <= hi; ++j) v = fmaxf(v, raw[j]);
    } else {
      v = 0.f;
      const int lo = max(i - h, 0), hi = min(i + h, E - 1);
      for (int j = lo; j <= hi; ++j) v += raw[j];
    }
    keys[i] = float_key(v);
    kr.add(keys[i], true);
  }
}

// Builds the keys of [0, E) and returns their range in sh.bcast (lo, hi).
__device__ void build_keys(uint32_t* keys, const float* raw, int E, int pool, int pool_type, bool do_pool,
                           bool aligned4, SelShared& sh) {
  const bool is_max = pool_type == KVEV_POOL_MAX;
  KeyRange kr;
  bool done = false;
  if (aligned4) {
    done = true;
    if (!do_pool) build_raw4(keys, raw, E, kr);
    else if (pool == 3) build_pooled4<3>(keys, raw, E, is_max, kr);
    else if (pool == 5) build_pooled4<5>(keys, raw, E, is_max, kr);
    else if (pool == 7) build_pooled4<7>(keys, raw, E, is_max, kr);
    else if (pool == 9) build_pooled4<9>(keys, raw, E, is_max, kr);
    else done = false;
  }
  if (!done) build_scalar(keys, raw, E, pool, do_pool, is_max, kr);
  const uint32_t lo = __reduce_min_sync(0xffffffffu, kr.lo), hi = __reduce_max_sync(0xffffffffu, kr.hi);
  if ((threadIdx.x & 31) == 0) {
    atomicMin(reinterpret_cast<unsigned*>(&sh.bcast[0]), lo);
    atomicMax(reinterpret_cast<unsigned*>(&sh.bcast[1]), hi);
  }
}

// Pass 2: histogram of the first digit (key - lo) >> s, which splits the keys'
// range into at most kBins0 bins of 2^s keys each (plain atomics: keys spread
// over the bins).
__device__ void range_hist(const uint32_t* keys, int E, uint32_t lo, int s, int* hist) {
  constexpr int R = kSelectUnroll;
  for (int b0 = 0; b0 < E; b0 += 4 * R * kSelectThreads) {
    uint4 kv[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + (r * kSelectThreads + threadIdx.x) * 4;
      kv[r] = i0 < E ? ld_keys4(keys, i0) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + (r * kSelectThreads + threadIdx.x) * 4;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u < E) atomicAdd(&hist[(pick(kv[r], u) - lo) >> s], 1);
    }
  }
}

// ---------------------------------------------------------------------------
// Pass 2 and the candidate radix passes.
// ---------------------------------------------------------------------------

// Each warp counts its segment's keys of first-digit bins above d (into wgt)
// and appends the keys of bin d, with their positions, to the candidate list
// (in no particular order; at most kCandCap are stored, ncand counts them all).
__device__ void collect_candidates(const uint32_t* keys, int E, uint32_t lo_key, int s, uint32_t d,
                                   SelShared& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int gt = 0;
  constexpr int R = kSelectUnroll;
  for (int b0 = lo; b0 < hi; b0 += R * kSegKeys) {
    uint4 kv[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + r * kSegKeys + 4 * lane;
      kv[r] = i0 < hi ? ld_keys4(keys, i0) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + r * kSegKeys + 4 * lane;
      int c = 0;
      uint32_t cmask = 0;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool valid = i0 + u < hi;
        const uint32_t q = (pick(kv[r], u) - lo_key) >> s;
        gt += valid && q > d;
        const bool in = valid && q == d;
        cmask |= static_cast<uint32_t>(in) << u;
        c += in;
      }
      if (__any_sync(0xffffffffu, c)) {
        const int incl = warp_incl(c);
        int base = 0;
        if (lane == 31) base = atomicAdd(&sh.ncand, incl);
        base = __shfl_sync(0xffffffffu, base, 31) + incl - c;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (cmask & (1u << u)) {
            if (base < kCandCap) sh.u.cand[base] = make_uint2(static_cast<uint32_t>(i0 + u), pick(kv[r], u));
            ++base;
          }
        }
      }
    }
  }
  gt = warp_sum(gt);
  if (lane == 0) {
    sh.wgt[warp] = gt;
    sh.weq[warp] = 0;
  }
}

// Threshold key T (the kk-th largest of the candidates, the keys of first-digit
// bin d) and how many keys equal to T to keep, by radix passes of up to 9 bits
// over the s low bits of key - lo_key; then each candidate above or equal to
// T is tallied to its warp segment.
__device__ void select_candidates(int E, uint32_t lo_key, int s, uint32_t d, int kk, SelShared& sh,
                                  uint32_t& T, int& need) {
  const int nc = sh.ncand;
  uint32_t prefix = 0, mask = 0;  // over the s low bits
  for (int r = s; r > 0;) {
    const int nb = min(9, r), shift = r - nb;
    const uint32_t dm = (1u << nb) - 1u;
    for (int i = threadIdx.x; i < kBins1; i += kSelectThreads) sh.hist1[i] = 0;
    __syncthreads();
    for (int c = threadIdx.x; c < nc; c += kSelectThreads) {
      const uint32_t v = sh.u.cand[c].y - lo_key;
      if ((v & mask) == prefix) atomicAdd(&sh.hist1[(v >> shift) & dm], 1);
    }
    __syncthreads();
    int digit, above;
    find_bin(sh.hist1, kBins1, kk, sh, digit, above);
    kk -= above;
    prefix |= static_cast<uint32_t>(digit) << shift;
    mask |= dm << shift;
    r = shift;
  }
  T = lo_key + ((d << s) | prefix);
  need = kk;
  const int seg = seg_len(E);
  for (int c = threadIdx.x; c < nc; c += kSelectThreads) {
    const uint2 e = sh.u.cand[c];
    const int w = static_cast<int>(e.x) / seg;
    if (e.y > T) atomicAdd(&sh.wgt[w], 1);
    else if (e.y == T) atomicAdd(&sh.weq[w], 1);
  }
  __syncthreads();
}

// The general path: four 8-bit radix passes over every key, then each warp
// counts its segment's keys above and equal to T.
__device__ void select_all_keys(const uint32_t* keys, int E, int k, SelShared& sh, uint32_t& T, int& need) {
  uint32_t prefix = 0, mask = 0;
  int kk = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += kSelectThreads) sh.hist1[i] = 0;
    __syncthreads();
    for (int b0 = 0; b0 < E; b0 += 4 * kSelectThreads) {
      const int i0 = b0 + 4 * threadIdx.x;
      const uint4 kv = i0 < E ? ld_keys4(keys, i0) : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t key = pick(kv, u);
        const bool in = i0 + u < E && (key & mask) == prefix;
        hist_add(sh.hist1, in, (key >> shift) & 255u);
      }
    }
    __syncthreads();
    int digit, above;
    find_bin(sh.hist1, 256, kk, sh, digit, above);
    kk -= above;
    prefix |= static_cast<uint32_t>(digit) << shift;
    mask |= 255u << shift;
  }
  T = prefix;
  need = kk;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int gt = 0, eq = 0;
  for (int b0 = lo; b0 < hi; b0 += kSegKeys) {
    const int i0 = b0 + 4 * lane;
    const uint4 kv = i0 < hi ? ld_keys4(keys, i0) : make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const bool valid = i0 + u < hi;
      gt += valid && pick(kv, u) > T;
      eq += valid && pick(kv, u) == T;
    }
  }
  gt = warp_sum(gt);
  eq = warp_sum(eq);
  if (lane == 0) {
    sh.wgt[warp] = gt;
    sh.weq[warp] = eq;
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Pass 4: ordered write of the kept positions of [0, E) to out[0..k): keys
// above T, and the first `need` keys equal to T in position order.
// ---------------------------------------------------------------------------
__device__ void write_kept(const uint32_t* keys, int E, int k, uint32_t T, int need, const SelShared& sh,
                           int* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int eq_base = 0, sel_base = 0;
  for (int w = 0; w < warp; ++w) {
    const int e = sh.weq[w];
    sel_base += sh.wgt[w] + min(max(need - eq_base, 0), e);
    eq_base += e;
  }
  constexpr int R = kSelectUnroll;
  for (int b0 = lo; b0 < hi; b0 += R * kSegKeys) {
    uint4 kr[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + r * kSegKeys + 4 * lane;
      kr[r] = i0 < hi ? ld_keys4(keys, i0) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i0 = b0 + r * kSegKeys + 4 * lane;
      const uint4 kv = kr[r];
      uint32_t gm = 0, em = 0;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool valid = i0 + u < hi;
        gm |= static_cast<uint32_t>(valid && pick(kv, u) > T) << u;
        em |= static_cast<uint32_t>(valid && pick(kv, u) == T) << u;
      }
      if (!__any_sync(0xffffffffu, gm | em)) continue;
      // ranks of the keys equal to T, in position order
      const int ce = __popc(em);
      const int ie = warp_incl(ce);
      int rank = eq_base + ie - ce;
      uint32_t sm = gm;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (em & (1u << u)) {
          if (rank < need) sm |= 1u << u;
          ++rank;
        }
      }
      const int cs = __popc(sm);
      const int is = warp_incl(cs);
      int slot = sel_base + is - cs;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (sm & (1u << u)) {
          if (slot < k) out[slot] = i0 + u;
          ++slot;
        }
      }
      eq_base += __shfl_sync(0xffffffffu, ie, 31);
      sel_base += __shfl_sync(0xffffffffu, is, 31);
    }
  }
}

__global__ void __launch_bounds__(kSelectThreads, kSelectCtasPerSm) select_kernel(const __grid_constant__ SelectParams p) {
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
  uint32_t* keys = p.keys + (static_cast<size_t>(ld.score_slot) * per_layer + rem) * p.key_stride;
  for (int i = threadIdx.x; i < kBins0; i += kSelectThreads) sh.u.hist[i] = 0;
  if (threadIdx.x == 0) {
    sh.bcast[0] = static_cast<int>(0xFFFFFFFFu);  // key range, as unsigned
    sh.bcast[1] = 0;
    sh.ncand = 0;
  }
  __syncthreads();
  const bool aligned4 = (reinterpret_cast<uintptr_t>(raw) & 15u) == 0 && (p.S_cap & 3) == 0;
  build_keys(keys, raw, E, p.pool_kernel, p.pool_type, ld.method == KVEV_SNAPKV, aligned4, sh);
  __syncthreads();
  const uint32_t klo = static_cast<uint32_t>(sh.bcast[0]), khi = static_cast<uint32_t>(sh.bcast[1]);
  if (klo == khi) {  // every key equal: the lowest positions win the ties
    for (int j = threadIdx.x; j < k; j += blockDim.x) idx[j] = j;
    return;
  }
  // first digit: (key - klo) >> s, at most kBins0 bins over the keys' range
  const int s_bits = max(0, 32 - __clz(static_cast<int>(khi - klo)) - 13);
  range_hist(keys, E, klo, s_bits, sh.u.hist);
  __syncthreads();
  int d, above;
  find_bin(sh.u.hist, kBins0, k, sh, d, above);  // ends with a barrier: hist may be overwritten
  collect_candidates(keys, E, klo, s_bits, static_cast<uint32_t>(d), sh);
  __syncthreads();
  uint32_t T;
  int need;
  if (sh.ncand <= kCandCap)
    select_candidates(E, klo, s_bits, static_cast<uint32_t>(d), k - above, sh, T, need);
  else  // a crowded bin: many equal keys
    select_all_keys(keys, E, k, sh, T, need);
  write_kept(keys, E, k, T, need, sh, idx);
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, int grid, cudaStream_t s) {
  if (grid == 0) return cudaSuccess;
  select_kernel<<<grid, kSelectThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
