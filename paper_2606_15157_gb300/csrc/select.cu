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
//   Streaming: keep [0, sink) plus the last `recent` positions (closed form);
//              this launch also copies those K/V rows into the packed cache
//              (they need no scores, and the selection leaves HBM mostly
//              idle), so the gather launch skips these layers.
//   b >= n   : keep every position.
// Top-k order: larger score first, equal scores keep the lower position.
// Output indices are ascending; unused slots hold -1.
//
// CTAs take the SnapKV / H2O units longest sequence first (the units of the
// longest sequence, then of the next one ...), so the long selections start
// early; the StreamingLLM and FULL units are spread evenly between them, so
// that the copies' HBM traffic overlaps the latency-bound selections.
//
// A unit takes a CTA of 256 threads, so that several units share an SM and
// one unit's barriers and round trips overlap another's passes.  Keys are an
// order-preserving uint32 image of the fp32 (pooled) scores.  The unit's row
// of a workspace array holds, between the two passes, each key's 16-bit bin
// (transposed in 256-position blocks, so that one 16-byte load gives a lane
// eight positions and a warp's ballots rank them by position); it stays in
// L2:
//   0. 1024 keys sampled at even strides give the bins: their range, widened
//      by half on either side, split into 8192 bins of 2^s keys (a unit's
//      scores may crowd into a few per cent of one octave, or spread over
//      many octaves: the range adapts the bins to either);
//   1. build the keys, store their bins and histogram them (the two end bins
//      also take every key outside the range);
//   2. with the bin d holding the k-th largest key found, each warp walks its
//      segment of the bins in order: keys of higher bins are kept for sure
//      and their positions are staged, in order, as 16-bit offsets at the
//      start of the segment's row; keys of bin d (the candidates) go to the
//      warp's list in shared memory with the count of sure positions before
//      them, and their keys are recomputed from the scores;
//   3. radix passes of up to 9 bits over the candidates fix the threshold key
//      T and how many keys equal to T to keep (ties keep the lower position);
//   4. every warp merges its staged positions and its kept candidates into
//      its share of the output, after the shares of the warps before it.
// An end bin, or a candidate list that overflows (many equal keys), takes the
// general path instead: the full keys are written to the row (transposed
// 128-key blocks), four 8-bit radix passes over every key fix T, and one
// ordered pass writes the kept positions.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

constexpr int kSW = kSelectThreads / 32;   // warps of a selection CTA
constexpr int kBins0 = 8192;               // bins of the sampled range
constexpr int kCandPerWarp = 320;          // candidates a warp's list holds
constexpr int kBins1 = 512;                // candidate digits: up to 9 bits a pass
constexpr int kSegKeys = 128;              // a key block: four keys per lane
constexpr int kBinBlock = 256;             // a bin block: eight positions per lane

struct CandLists {
  uint32_t pos[kSW][kCandPerWarp];
  uint32_t key[kSW][kCandPerWarp];
  int sure[kSW][kCandPerWarp];  // sure positions of the segment before the candidate
};

struct __align__(16) SelShared {
  union {
    int hist[kBins0];
    CandLists c;
  } u;
  int hist1[kBins1];
  int wsum[kSW];
  int wS[kSW];    // per warp segment: sure positions staged
  int wC[kSW];    // per warp segment: candidates
  int wgt[kSW];   // per warp segment: keys above T (general path) / candidates above T
  int weq[kSW];   // per warp segment: keys (candidates) equal to T
  int bcast[2];
  uint32_t rlo, rhi;  // sampled key range, then the candidates' key range
  int overflow;
};

static_assert(sizeof(SelShared) <= 48 * 1024, "the selection's shared memory is static");
static_assert(sizeof(CandLists) <= sizeof(int) * kBins0, "the candidate lists reuse the histogram");

// Adds each valid lane's digit to the histogram, one shared-memory atomic per
// distinct digit of the warp (for digits that crowd into few bins).  Every
// lane of the warp must call it.
__device__ __forceinline__ void hist_add(int* hist, bool valid, uint32_t digit) {
  const uint32_t d = valid ? digit : 0xFFFFFFFFu;
  const uint32_t peers = __match_any_sync(0xffffffffu, d);
  if (valid && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[d], __popc(peers));
}

// The first digit: the bin of the key within [lo, lo + 8192 * 2^s); keys
// below or above the range fall into the end bins.
struct Binning {
  uint32_t lo;
  int s;
  __device__ __forceinline__ uint32_t bin(uint32_t key) const {
    return key < lo ? 0u : min((key - lo) >> s, static_cast<uint32_t>(kBins0 - 1));
  }
};

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

// Warp segments of [0, E): contiguous, whole 256-position blocks, in warp
// order, so that a warp's kept positions follow those of the warps before it.
__device__ __forceinline__ int seg_len(int E) {
  return ((E + kSW - 1) / kSW + kBinBlock - 1) / kBinBlock * kBinBlock;
}

__device__ __forceinline__ uint32_t pick(const uint4& v, int u) {
  return u == 0 ? v.x : u == 1 ? v.y : u == 2 ? v.z : v.w;
}

// A key row holds 128-key blocks, each transposed: the key of position
// b + 32u + L (b a multiple of 128, L < 32, u < 4) sits at b + 4L + u, so that
// one 16-byte load gives lane L its four keys of the block in position order
// and a ballot per u ranks a warp's keys by position.  Rows are padded to
// whole blocks.
__device__ __forceinline__ int tpos(int i) { return (i & ~127) | ((i & 31) << 2) | ((i >> 5) & 3); }

// Lane L's four keys of the block at b0: positions b0 + L + 32u.
__device__ __forceinline__ uint4 ld_block_keys(const uint32_t* keys, int b0) {
  return __ldcg(reinterpret_cast<const uint4*>(keys + b0 + 4 * (threadIdx.x & 31)));
}

// The fast path keeps 16-bit bins instead of keys, in 256-position blocks
// transposed the same way: the bin of position b + 32u + L (u < 8) sits at
// 16-bit index b + 8L + u, so one 16-byte load gives lane L eight positions.
__device__ __forceinline__ int tpos16(int i) { return (i & ~255) | ((i & 31) << 3) | ((i >> 5) & 7); }

__device__ __forceinline__ uint4 ld_block_bins(const uint16_t* bins, int b0) {
  return __ldcg(reinterpret_cast<const uint4*>(bins + b0 + 8 * (threadIdx.x & 31)));
}

__device__ __forceinline__ uint32_t pick16(const uint4& v, int u) {
  const uint32_t w = pick(v, u >> 1);
  return (u & 1) ? (w >> 16) : (w & 0xFFFFu);
}


// Bulk prefetch of the floats [src, src + n) into L2, in 16 KiB pieces, one
// per thread (the row is 16-byte aligned and padded to whole 16-byte blocks).
__device__ __forceinline__ void prefetch_row_l2(const float* src, int n) {
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(src);
  const uintptr_t a1 = (reinterpret_cast<uintptr_t>(src + n) + 15) & ~uintptr_t(15);
  for (uintptr_t a = a0 + static_cast<uintptr_t>(threadIdx.x) * 16384; a < a1; a += 16384u * kSelectThreads) {
    const uint32_t bytes = static_cast<uint32_t>(a1 - a < 16384 ? a1 - a : 16384);
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(a), "r"(bytes) : "memory");
  }
}

// ---------------------------------------------------------------------------
// Key generators: four consecutive keys of [0, E) from position i0 (a multiple
// of four, i0 < E), in two halves -- load() issues the reads, keys() computes
// -- so that a pass can have the next block's reads in flight while it works
// on the current one.  Keys past E are computed but never used.
// ---------------------------------------------------------------------------

// Pooled keys from a 16-byte aligned score row (S_cap a multiple of 4): keys
// i0 .. i0+3 have windows (P <= 9) inside the three aligned 4-float chunks
// starting at i0 - 4, i0 and i0 + 4.  Only chunks that start before E are
// read (none leaves the row); entries outside [0, E) count as -inf (max) or 0
// (avg).  Avg pooling divides every window sum by the same p, so the sum
// ranks the keys alike and is used instead.
template <int P>
struct Pooled4 {
  const float* raw;
  int E;
  bool is_max;
  struct Regs {
    float4 c[3];
  };
  __device__ __forceinline__ void load(int i0, Regs& r) const {
    const float fill = is_max ? -INFINITY : 0.f;
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const int st = i0 - 4 + 4 * c;
      r.c[c] = make_float4(fill, fill, fill, fill);
      if (st >= 0 && st < E) r.c[c] = __ldg(reinterpret_cast<const float4*>(raw + st));  // neighbours': L1
    }
  }
  __device__ __forceinline__ void keys(int i0, const Regs& r, uint32_t (&kq)[4]) const {
    constexpr int h = P / 2;
    static_assert(h <= 4, "the three chunks cover windows of up to 9");
    float w[12];
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      w[4 * c + 0] = r.c[c].x;
      w[4 * c + 1] = r.c[c].y;
      w[4 * c + 2] = r.c[c].z;
      w[4 * c + 3] = r.c[c].w;
    }
    if (i0 + 8 > E) {  // the last chunk may run past E
      const float fill = is_max ? -INFINITY : 0.f;
#pragma unroll
      for (int j = 0; j < 12; ++j)
        if (i0 - 4 + j >= E) w[j] = fill;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      float v = w[4 + u - h];
#pragma unroll
      for (int j = 1; j < P; ++j) v = is_max ? fmaxf(v, w[4 + u - h + j]) : v + w[4 + u - h + j];
      kq[u] = float_key(v);
    }
  }
};

// Raw keys (no pooling) from a 16-byte aligned score row.
struct Raw4 {
  const float* raw;
  int E;
  struct Regs {
    float4 v;
  };
  __device__ __forceinline__ void load(int i0, Regs& r) const {
    r.v = __ldg(reinterpret_cast<const float4*>(raw + i0));
  }
  __device__ __forceinline__ void keys(int, const Regs& r, uint32_t (&kq)[4]) const {
    kq[0] = float_key(r.v.x);
    kq[1] = float_key(r.v.y);
    kq[2] = float_key(r.v.z);
    kq[3] = float_key(r.v.w);
  }
};

// Any alignment and any odd pooling width: scalar loads, all in keys().
struct Scalar4 {
  const float* raw;
  int E, h;
  bool do_pool, is_max;
  struct Regs {};
  __device__ __forceinline__ uint32_t one(int i) const {
    if (!do_pool) return float_key(raw[i]);
    const int lo = max(i - h, 0), hi = min(i + h, E - 1);
    float v = is_max ? -INFINITY : 0.f;
    for (int j = lo; j <= hi; ++j) v = is_max ? fmaxf(v, raw[j]) : v + raw[j];
    return float_key(v);
  }
  __device__ __forceinline__ void load(int, Regs&) const {}
  __device__ __forceinline__ void keys(int i0, const Regs&, uint32_t (&kq)[4]) const {
#pragma unroll
    for (int u = 0; u < 4; ++u) kq[u] = i0 + u < E ? one(i0 + u) : 0u;
  }
};

template <class Gen>
__device__ __forceinline__ void gen_keys(const Gen& gen, int i0, uint32_t (&kq)[4]) {
  typename Gen::Regs r;
  gen.load(i0, r);
  gen.keys(i0, r, kq);
}

// ---------------------------------------------------------------------------
// Step 0: the bracket.  Sample keys: thread t takes the group of four at
// 4 * floor(t * ceil(E / 4) / 256).  Their range is widened by half of it on
// either side (at least 4096 key steps) and split into 8192 bins.
// ---------------------------------------------------------------------------
__device__ __forceinline__ Binning make_binning(uint32_t a, uint32_t b) {
  const uint32_t m = max((b - a) / 2u, 4096u);
  const uint32_t lo = a > m ? a - m : 0u;
  const uint32_t hi = 0xFFFFFFFFu - b > m ? b + m : 0xFFFFFFFFu;
  Binning bn;
  bn.lo = lo;
  bn.s = max(0, 32 - __clz(static_cast<int>(hi - lo)) - 13);  // (hi - lo) >> s < 8192
  return bn;
}

struct Bracket {
  Binning bn;
  uint32_t lo_bin, hi_bin;  // candidates: bins lo_bin .. hi_bin; sure: bins above hi_bin
};

// The binning of the unit's keys from its sample.  Needs sh.rlo / sh.rhi
// initialised.
template <class Gen>
__device__ Binning sample_binning(const Gen& gen, int E, SelShared& sh) {
  const int groups = (E + 3) / 4;
  const int i0 = 4 * static_cast<int>((static_cast<long long>(threadIdx.x) * groups) / kSelectThreads);
  uint32_t kq[4];
  gen_keys(gen, i0, kq);
  uint32_t lo = 0xFFFFFFFFu, hi = 0u;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    if (i0 + u < E) {
      lo = min(lo, kq[u]);
      hi = max(hi, kq[u]);
    }
  }
  lo = __reduce_min_sync(0xffffffffu, lo);
  hi = __reduce_max_sync(0xffffffffu, hi);
  if ((threadIdx.x & 31) == 0) {
    atomicMin(&sh.rlo, lo);
    atomicMax(&sh.rhi, hi);
  }
  __syncthreads();
  return make_binning(sh.rlo, sh.rhi);
}

// Step 1: the bin of every key of [0, E) into the unit's workspace row (16-bit
// transposed blocks), and the histogram of the bins.
template <class Gen>
__device__ void build_row_hist(const Gen& gen, uint16_t* bins, int E, Binning bn, int* hist) {
  typename Gen::Regs nxt;
  int i0 = 4 * threadIdx.x;
  if (i0 < E) gen.load(i0, nxt);
  for (; i0 < E; i0 += 4 * kSelectThreads) {
    const typename Gen::Regs cur = nxt;
    if (i0 + 4 * kSelectThreads < E) gen.load(i0 + 4 * kSelectThreads, nxt);  // next reads go out first
    uint32_t kq[4];
    gen.keys(i0, cur, kq);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (i0 + u < E) {
        const uint32_t b = bn.bin(kq[u]);
        bins[tpos16(i0 + u)] = static_cast<uint16_t>(b);
        atomicAdd(&hist[b], 1);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Step 2: each warp walks its segment [lo, hi) of the bins in order.  Keys of
// bins above the bracket are kept for sure: their positions are staged, in
// order, as 16-bit offsets at the start of the segment's row (a warp only
// overwrites entries of positions it has passed, and has the next block's
// bins in registers).  Keys inside the bracket (the candidates) go to the
// warp's list with the count of sure positions before them; their keys are
// recomputed from the scores afterwards.  A list that fills up sets
// sh.overflow.
// ---------------------------------------------------------------------------
__device__ void classify_pass(uint16_t* bins, int E, const Bracket& br, SelShared& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int ns = 0, nc = 0;  // sure positions staged, candidates listed
  uint4 nxt = make_uint4(0, 0, 0, 0);
  if (lo < hi) nxt = ld_block_bins(bins, lo);
  for (int b0 = lo; b0 < hi; b0 += kBinBlock) {
    const uint4 cur = nxt;
    if (b0 + kBinBlock < hi) nxt = ld_block_bins(bins, b0 + kBinBlock);  // the next block goes out first
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int p = b0 + 32 * u + lane;
      const uint32_t q = pick16(cur, u);
      const bool valid = p < hi;
      const bool sure = valid && q > br.hi_bin;
      const bool cand = valid && q >= br.lo_bin && q <= br.hi_bin;
      const uint32_t bs = __ballot_sync(0xffffffffu, sure), bc = __ballot_sync(0xffffffffu, cand);
      const int js = ns + __popc(bs & lt);
      // staged as offsets from the segment start, behind the positions already read
      if (sure) bins[lo + js] = static_cast<uint16_t>(p - lo);
      if (cand) {
        const int jc = nc + __popc(bc & lt);
        if (jc < kCandPerWarp) {
          sh.u.c.pos[warp][jc] = static_cast<uint32_t>(p);
          sh.u.c.sure[warp][jc] = js;
        }
      }
      ns += __popc(bs);
      nc += __popc(bc);
    }
  }
  if (lane == 0) {
    sh.wS[warp] = ns;
    sh.wC[warp] = nc;
    if (nc > kCandPerWarp) sh.overflow = 1;
  }
}

// The keys of each warp's listed candidates, from the scores.
__device__ void candidate_keys(const Scalar4& sk, SelShared& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nc = min(sh.wC[warp], kCandPerWarp);
  for (int i = lane; i < nc; i += 32) sh.u.c.key[warp][i] = sk.one(static_cast<int>(sh.u.c.pos[warp][i]));
}

// Step 3: threshold key T (the kk-th largest candidate) and how many keys
// equal to T to keep, by radix passes of up to 9 bits over key - (least
// candidate key); then each warp counts its candidates above and equal to T.
__device__ void select_candidates(int kk, SelShared& sh, uint32_t& T, int& need) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    sh.rlo = 0xFFFFFFFFu;
    sh.rhi = 0u;
  }
  __syncthreads();
  uint32_t lo = 0xFFFFFFFFu, hi = 0u;
  for (int i = lane; i < sh.wC[warp]; i += 32) {
    lo = min(lo, sh.u.c.key[warp][i]);
    hi = max(hi, sh.u.c.key[warp][i]);
  }
  lo = __reduce_min_sync(0xffffffffu, lo);
  hi = __reduce_max_sync(0xffffffffu, hi);
  if (lane == 0) {
    atomicMin(&sh.rlo, lo);
    atomicMax(&sh.rhi, hi);
  }
  __syncthreads();
  const uint32_t clo = sh.rlo, span = sh.rhi - sh.rlo;
  const int bits = span == 0 ? 0 : 32 - __clz(static_cast<int>(span));
  uint32_t prefix = 0, mask = 0;  // over the low `bits` bits of key - clo
  for (int r = bits; r > 0;) {
    const int nb = min(9, r), shift = r - nb;
    const uint32_t dm = (1u << nb) - 1u;
    for (int i = threadIdx.x; i < kBins1; i += kSelectThreads) sh.hist1[i] = 0;
    __syncthreads();
    for (int c = threadIdx.x; c < kSW * kCandPerWarp; c += kSelectThreads) {
      const int w = c / kCandPerWarp, i = c - w * kCandPerWarp;
      if (i < sh.wC[w]) {
        const uint32_t v = sh.u.c.key[w][i] - clo;
        if ((v & mask) == prefix) atomicAdd(&sh.hist1[(v >> shift) & dm], 1);
      }
    }
    __syncthreads();
    int digit, above;
    find_bin(sh.hist1, kBins1, kk, sh, digit, above);
    kk -= above;
    prefix |= static_cast<uint32_t>(digit) << shift;
    mask |= dm << shift;
    r = shift;
  }
  T = clo + prefix;
  need = kk;
  int gt = 0, eq = 0;
  for (int i = lane; i < sh.wC[warp]; i += 32) {
    const uint32_t key = sh.u.c.key[warp][i];
    gt += key > T;
    eq += key == T;
  }
  gt = warp_sum(gt);
  eq = warp_sum(eq);
  if (lane == 0) {
    sh.wgt[warp] = gt;
    sh.weq[warp] = eq;
  }
  __syncthreads();
}

// Step 4: warp w's output share starts after the shares (sure positions plus
// kept candidates) of the warps before it.  Its kept candidates go to
// base + (sure positions before it) + (kept candidates before it); its sure
// position j to base + j + (kept candidates with at most j sure positions
// before them).
__device__ void merge_write(const uint16_t* bins, int E, int k, int need, SelShared& sh, uint32_t T, int* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  int base = 0, eq_base = 0;
  for (int w = 0; w < warp; ++w) {
    base += sh.wS[w] + sh.wgt[w] + min(max(need - eq_base, 0), sh.weq[w]);
    eq_base += sh.weq[w];
  }
  const int nc = sh.wC[warp];
  int* sure = sh.u.c.sure[warp];
  int nk = 0;  // kept candidates so far; their sure counts are compacted into sure[0 .. nk)
  for (int i0 = 0; i0 < nc; i0 += 32) {
    const int i = i0 + lane;
    uint32_t key = 0, pos = 0;
    int sb = 0;
    if (i < nc) {
      key = sh.u.c.key[warp][i];
      pos = sh.u.c.pos[warp][i];
      sb = sure[i];
    }
    const bool e = i < nc && key == T;
    const uint32_t eb = __ballot_sync(0xffffffffu, e);
    const bool keep = i < nc && (key > T || (e && eq_base + __popc(eb & lt) < need));
    const uint32_t kb = __ballot_sync(0xffffffffu, keep);
    const int ki = nk + __popc(kb & lt);
    __syncwarp();  // every lane has read its entry before the compaction overwrites it
    if (keep) {
      if (base + sb + ki < k) out[base + sb + ki] = static_cast<int>(pos);
      sure[ki] = sb;
    }
    __syncwarp();
    nk += __popc(kb);
    eq_base += __popc(eb);
  }
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E);
  const int ns = sh.wS[warp];
  for (int j = lane; j < ns; j += 32) {
    const int pos = lo + static_cast<int>(__ldcg(bins + lo + j));
    int a = 0, b = nk;  // kept candidates with sure[] <= j: the first index with sure[] > j
    while (a < b) {
      const int m = (a + b) >> 1;
      if (sure[m] <= j) a = m + 1;
      else b = m;
    }
    if (base + j + a < k) out[base + j + a] = pos;
  }
}

// The general path: four 8-bit radix passes over every key, then each warp
// counts its segment's keys above and equal to T.
__device__ void select_all_keys(const uint32_t* keys, int E, int k, SelShared& sh, uint32_t& T, int& need) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t prefix = 0, mask = 0;
  int kk = k;
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += kSelectThreads) sh.hist1[i] = 0;
    __syncthreads();
    for (int b0 = 128 * warp; b0 < E; b0 += 128 * kSW) {  // blocks dealt to the warps in turn
      const uint4 kv = ld_block_keys(keys, b0);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t key = pick(kv, u);
        const bool in = b0 + 32 * u + lane < E && (key & mask) == prefix;
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
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int gt = 0, eq = 0;
  for (int b0 = lo; b0 < hi; b0 += kSegKeys) {
    const uint4 kv = ld_block_keys(keys, b0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const bool valid = b0 + 32 * u + lane < hi;
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
// The general path's ordered write of the kept positions of [0, E) to
// out[0..k): keys above T, and the first `need` keys equal to T in position
// order.
// ---------------------------------------------------------------------------
__device__ void write_kept(const uint32_t* keys, int E, int k, uint32_t T, int need, const SelShared& sh,
                           int* out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  const int seg = seg_len(E);
  const int lo = min(warp * seg, E), hi = min(lo + seg, E);
  int eq_base = 0, sel_base = 0;
  for (int w = 0; w < warp; ++w) {
    const int e = sh.weq[w];
    sel_base += sh.wgt[w] + min(max(need - eq_base, 0), e);
    eq_base += e;
  }
  for (int b0 = lo; b0 < hi; b0 += kSegKeys) {
    const uint4 kv = ld_block_keys(keys, b0);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int p = b0 + 32 * u + lane;
      const bool valid = p < hi;
      const bool g = valid && pick(kv, u) > T, e = valid && pick(kv, u) == T;
      const uint32_t be = __ballot_sync(0xffffffffu, e);
      const bool sel = g || (e && eq_base + __popc(be & lt) < need);
      const uint32_t bsel = __ballot_sync(0xffffffffu, sel);
      const int slot = sel_base + __popc(bsel & lt);
      if (sel && slot < k) out[slot] = p;
      eq_base += __popc(be);
      sel_base += __popc(bsel);
    }
  }
}

// Every key of [0, E) into the unit's workspace row, transposed blocks (the
// general path).
template <class Gen>
__device__ void build_row(const Gen& gen, uint32_t* row, int E) {
  for (int i0 = 4 * threadIdx.x; i0 < E; i0 += 4 * kSelectThreads) {
    uint32_t kq[4];
    gen_keys(gen, i0, kq);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (i0 + u < E) row[tpos(i0 + u)] = kq[u];
  }
}

// Top-k of the keys of [0, E) (1 <= k < E) into out[0 .. k), ascending.
template <class Gen>
__device__ void select_unit(const Gen& gen, const Scalar4& sk, uint32_t* row, int E, int k, SelShared& sh,
                            int* out) {
  for (int i = threadIdx.x; i < kBins0; i += kSelectThreads) sh.u.hist[i] = 0;
  if (threadIdx.x == 0) {
    sh.rlo = 0xFFFFFFFFu;
    sh.rhi = 0u;
    sh.overflow = 0;
  }
  __syncthreads();
  const Binning bn = sample_binning(gen, E, sh);
  uint16_t* bins = reinterpret_cast<uint16_t*>(row);
  build_row_hist(gen, bins, E, bn, sh.u.hist);
  __syncthreads();
  int d, above;
  find_bin(sh.u.hist, kBins0, k, sh, d, above);  // ends with a barrier
  const int nd = sh.u.hist[d];
  __syncthreads();  // every thread has read it before the candidate lists overwrite the histogram
  // the end bins also hold keys outside the sampled range: not one prefix
  bool fast = d > 0 && d < kBins0 - 1 && nd <= kSW * kCandPerWarp && seg_len(E) <= 65536;
  if (fast) {
    const Bracket br{bn, static_cast<uint32_t>(d), static_cast<uint32_t>(d)};
    classify_pass(bins, E, br, sh);
    __syncthreads();
    fast = !sh.overflow;
    if (fast) {
      candidate_keys(sk, sh);
      __syncthreads();
    }
  }
  uint32_t T;
  int need;
  if (fast) {
    select_candidates(k - above, sh, T, need);
    merge_write(bins, E, k, need, sh, T, out);
    return;
  }
  // the general path: many equal keys, or a sample that missed the k-th key:
  // the row holds bins, so the keys are built now
  build_row(gen, row, E);
  __syncthreads();
  select_all_keys(row, E, k, sh, T, need);
  write_kept(row, E, k, T, need, sh, out);
}

// The sequence of rank r in order of decreasing length (equal lengths: lower
// index first), by warp 0 (B <= 32; larger batches keep the index order).
__device__ int seq_of_rank(const SelectParams& p, int r, SelShared& sh) {
  if (p.B > 32) return r;
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    const int n = lane < p.B ? p.lens[lane] : -1;
    int rank = 0;
    for (int j = 0; j < p.B; ++j) {
      const int nj = __shfl_sync(0xffffffffu, n, j);
      rank += nj > n || (nj == n && j < lane);
    }
    const uint32_t m = __ballot_sync(0xffffffffu, lane < p.B && rank == r);
    if (lane == 0) sh.bcast[0] = __ffs(m) - 1;
  }
  __syncthreads();
  return sh.bcast[0];
}

// A StreamingLLM unit's kept rows (positions pos_j of slots j < count) into its
// packed output rows, K and V as 16-byte vectors, four of each in flight per
// thread; slots past the count are zero-filled.
__device__ void copy_streaming_rows(const SelectParams& p, int l, int rem, int n, int count, bool identity) {
  const LayerDesc& ld = p.layer[l];
  const int vec = p.d / 8, total = ld.slots * vec;
  const size_t src0 = static_cast<size_t>(rem) * p.S_cap * vec;
  const size_t dst0 = (static_cast<size_t>(ld.row_off) + static_cast<size_t>(rem) * ld.slots) * vec;
  const uint4* Ks = static_cast<const uint4*>(p.K[l]) + src0;
  const uint4* Vs = static_cast<const uint4*>(p.V[l]) + src0;
  uint4* Kd = static_cast<uint4*>(p.out_K) + dst0;
  uint4* Vd = static_cast<uint4*>(p.out_V) + dst0;
  constexpr int kU = 4;
  for (int i0 = threadIdx.x; i0 < total; i0 += kU * kSelectThreads) {
    uint4 kv[kU], vv[kU];
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int i = i0 + q * kSelectThreads;
      kv[q] = make_uint4(0, 0, 0, 0);
      vv[q] = make_uint4(0, 0, 0, 0);
      const int j = i / vec;
      if (i < total && j < count) {
        const int pos = identity || j < p.sink ? j : n - ld.recent + (j - p.sink);
        const size_t e = static_cast<size_t>(pos) * vec + (i - j * vec);
        kv[q] = __ldg(Ks + e);
        vv[q] = __ldg(Vs + e);
      }
    }
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int i = i0 + q * kSelectThreads;
      if (i < total) {
        __stcs(Kd + i, kv[q]);
        __stcs(Vd + i, vv[q]);
      }
    }
  }
}

__global__ void __launch_bounds__(kSelectThreads, kSelectCtasPerSm) select_kernel(const __grid_constant__ SelectParams p) {
  __shared__ SelShared sh;
  const int per_layer = p.B * p.H_kv;
  // dispatch order: two lists, each in (sequence rank, layer, head) order --
  // the first L_first layers of p.order (the scoring layers) and the rest --
  // merged evenly: CTA b takes the c-th unit of the second list when
  // c = floor(b n2 / N) steps up at b, else the (b - c)-th of the first
  const long long N = static_cast<long long>(p.L) * per_layer;
  const long long n2 = static_cast<long long>(p.L - p.L_first) * per_layer;
  const int c = static_cast<int>(blockIdx.x * n2 / N);
  const bool second = (blockIdx.x + 1) * n2 / N > c;
  int b = second ? c : static_cast<int>(blockIdx.x) - c;
  const int first = second ? p.L_first : 0;
  const int nl = second ? p.L - p.L_first : p.L_first;
  const int r = b / (nl * p.H_kv);
  const int t = b - r * nl * p.H_kv;
  const int l = p.order[first + t / p.H_kv];
  const int h = t - (t / p.H_kv) * p.H_kv;
  const int s = seq_of_rank(p, r, sh);
  const int rem = s * p.H_kv + h;
  const LayerDesc ld = p.layer[l];
  const int n = p.lens[s];
  int* cnt = p.out_count + static_cast<size_t>(l) * per_layer + rem;
  if (ld.method == KVEV_FULL) {
    if (threadIdx.x == 0) *cnt = n;
    return;
  }
  const int b_l = ld.slots;
  int* idx = p.out_idx + ld.row_off + static_cast<long long>(rem) * b_l;

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
    copy_streaming_rows(p, l, rem, n, count, identity);
  } else {
    identity = n <= b_l;
    count = identity ? n : b_l;
    if (!identity) {
      const int protect = ld.method == KVEV_SNAPKV ? p.W : ld.h2o_recent;
      E = n - protect;
      k = b_l - protect;
    }
  }
  if (identity)
    for (int j = threadIdx.x; j < n; j += blockDim.x) idx[j] = j;
  for (int j = count + threadIdx.x; j < b_l; j += blockDim.x) idx[j] = -1;
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
  uint32_t* row = p.keys + (static_cast<size_t>(ld.score_slot) * per_layer + rem) * p.key_stride;
  const bool do_pool = ld.method == KVEV_SNAPKV, is_max = p.pool_type == KVEV_POOL_MAX;
  const bool aligned4 = (reinterpret_cast<uintptr_t>(raw) & 15u) == 0 && (p.S_cap & 3) == 0;
  if (aligned4) prefetch_row_l2(raw, E);  // the passes' score reads become L2 hits
  const Scalar4 sk{raw, E, p.pool_kernel / 2, do_pool, is_max};  // one key at a time (candidates)
  if (aligned4 && !do_pool) return select_unit(Raw4{raw, E}, sk, row, E, k, sh, idx);
  if (aligned4) {
    switch (p.pool_kernel) {
      case 3: return select_unit(Pooled4<3>{raw, E, is_max}, sk, row, E, k, sh, idx);
      case 5: return select_unit(Pooled4<5>{raw, E, is_max}, sk, row, E, k, sh, idx);
      case 7: return select_unit(Pooled4<7>{raw, E, is_max}, sk, row, E, k, sh, idx);
      case 9: return select_unit(Pooled4<9>{raw, E, is_max}, sk, row, E, k, sh, idx);
      default: break;
    }
  }
  select_unit(sk, sk, row, E, k, sh, idx);
}

}  // namespace

cudaError_t launch_select(const SelectParams& p, int grid, cudaStream_t s) {
  if (grid == 0) return cudaSuccess;
  select_kernel<<<grid, kSelectThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
