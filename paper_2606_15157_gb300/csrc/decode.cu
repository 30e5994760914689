// decode.cu -- decode-phase update of the retained caches, one generated token
// per call, for every layer of a route in one launch (the decode step of the
// rules Sec. 2.1 cites: H2O accumulates the new token's attention, TOVA keeps
// only the current step's attention, StreamingLLM keeps sinks + a rolling
// window, and a layer without a decode-phase rule appends).
//
// Decode arena (caller-owned device memory, layout from the plan): layer l
// holds B*H_kv*cap_l slots, slot (s, h, j) at row row_off(l) + (s*H_kv + h) *
// cap_l + j of dec_K / dec_V.  The state buffer holds lens[B], and per unit u
// = unit_off(l) + s*H_kv + h: count[u], evicted[u], and per slot pos (the
// position it holds, -1 = empty) and acc (H2O: accumulated attention; TOVA:
// the last step's attention).  Slot order carries no meaning: an evicted
// slot is overwritten by the new token.
//
// One CTA per H2O / TOVA unit, and one warp per StreamingLLM or append-only
// unit (eight per CTA).  H2O / TOVA: the G query rows of the new token attend to
// every retained slot and to the new token, p_j = (1/G) sum_g softmax_j(q_g .
// k_j / sqrt(d)); acc += p (H2O) or acc = p (TOVA).  When the unit already
// holds b slots, the slot with the smallest acc among positions older than
// the protected recent window (r = h2o_recent for H2O, 0 for TOVA) is
// evicted, ties to the higher position, and the new token takes its place
// (unless the new token itself is the one evicted).  The retained K rows are
// streamed once, as 16-byte loads feeding m16n8k16 tensor-core products of
// the G query rows; logits stay in shared memory.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

constexpr int kDecodeThreads = 256;


// Unit index -> layer: the last layer whose first unit is <= u (layers
// without slots own no units and share their unit_off with the next layer).
__device__ __forceinline__ int find_dec_layer(const DecodeParams& p, int u) {
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.layer[mid].unit_off <= u) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

struct DecShared {
  float f[kDecodeThreads / 32];
  int i[2 * (kDecodeThreads / 32)];
  float g[8][kDecodeThreads / 32];  // per-head partials of the G <= 8 query heads
};

// Block-wide max (kMax) or sum of G values per thread, all heads in one
// exchange: warp shuffles, then one shared-memory round.
template <int G, bool kMax>
__device__ __forceinline__ void block_reduce_heads(float (&v)[G], DecShared& sh) {
#pragma unroll
  for (int g = 0; g < G; ++g)
    for (int o = 16; o > 0; o >>= 1) {
      const float y = __shfl_xor_sync(0xffffffffu, v[g], o);
      v[g] = kMax ? fmaxf(v[g], y) : v[g] + y;
    }
  __syncthreads();
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int g = 0; g < G; ++g) sh.g[g][threadIdx.x >> 5] = v[g];
  __syncthreads();
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float r = sh.g[g][0];
    for (int w = 1; w < kDecodeThreads / 32; ++w) r = kMax ? fmaxf(r, sh.g[g][w]) : r + sh.g[g][w];
    v[g] = r;
  }
}

// Eviction order: smaller key first, then higher position first.
__device__ __forceinline__ bool evict_before(float a, int pa, float b, int pb) {
  return a < b || (a == b && pa > pb);
}

// Block-wide first candidate in eviction order (candidates have pos >= 0);
// returns its slot, -1 if there is none.
__device__ __forceinline__ int block_evict_choice(float a, int pos, int slot, DecShared& sh) {
  for (int o = 16; o > 0; o >>= 1) {
    const float a2 = __shfl_xor_sync(0xffffffffu, a, o);
    const int p2 = __shfl_xor_sync(0xffffffffu, pos, o);
    const int s2 = __shfl_xor_sync(0xffffffffu, slot, o);
    if (p2 >= 0 && (pos < 0 || evict_before(a2, p2, a, pos))) {
      a = a2;
      pos = p2;
      slot = s2;
    }
  }
  __syncthreads();
  if ((threadIdx.x & 31) == 0) {
    const int w = threadIdx.x >> 5;
    sh.f[w] = a;
    sh.i[2 * w] = pos;
    sh.i[2 * w + 1] = slot;
  }
  __syncthreads();
  float ba = sh.f[0];
  int bp = sh.i[0], bs = sh.i[1];
  for (int i = 1; i < kDecodeThreads / 32; ++i) {
    const int pi = sh.i[2 * i];
    if (pi >= 0 && (bp < 0 || evict_before(sh.f[i], pi, ba, bp))) {
      ba = sh.f[i];
      bp = pi;
      bs = sh.i[2 * i + 1];
    }
  }
  return bp < 0 ? -1 : bs;
}

// Copy one d-wide bf16 row (16-byte vectors) with the whole block.
__device__ __forceinline__ void copy_row(uint16_t* dst, const uint16_t* src, int d) {
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x)
    reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
}

struct UnitRef {
  int l, s, h, u;
  size_t rows0;  // first slot row of the unit
};

// Put the new token into slot dst (its K/V row, position n, key acc_new) and
// finish the unit's bookkeeping.  Called by the whole block.
__device__ __forceinline__ void place_new(const DecodeParams& p, const UnitRef& r, int D, int dst, int n,
                                          float acc_new, int new_count, int evicted_pos) {
  if (dst >= 0) {
    const size_t src = static_cast<size_t>(r.s) * p.H_kv + r.h;
    copy_row(static_cast<uint16_t*>(p.K) + (r.rows0 + dst) * D,
             static_cast<const uint16_t*>(p.k_new[r.l]) + src * D, D);
    copy_row(static_cast<uint16_t*>(p.V) + (r.rows0 + dst) * D,
             static_cast<const uint16_t*>(p.v_new[r.l]) + src * D, D);
  }
  if (threadIdx.x == 0) {
    if (dst >= 0) {
      p.pos[r.rows0 + dst] = n;
      p.acc[r.rows0 + dst] = acc_new;
    }
    p.count[r.u] = new_count;
    p.evicted[r.u] = evicted_pos;
  }
}

// One m16n8k16 bf16 tensor-core product with fp32 accumulation (per warp):
// d[16 x 8] += a[16 x 16] * b[16 x 8].
__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Logits (base 2) of the G query rows against slots 0..c-1 and the new token
// (index c) into lg[head][j].
template <int D, int G>
__device__ __forceinline__ void unit_logits(const DecodeParams& p, const uint16_t* Kb, const uint16_t* qn,
                                            const uint16_t* kn, int c, int ld, float* lg) {
  constexpr int KP = D / 32;  // k-step pairs
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, tig = lane & 3;
  // B fragments: head gid (column), dims kp*32 + tig*8 + 4w + [0, 4) of k-step 2kp + w
  uint32_t bq[2 * KP][2];
#pragma unroll
  for (int kp = 0; kp < KP; ++kp) {
#pragma unroll
    for (int w = 0; w < 2; ++w) {
      uint2 v = make_uint2(0, 0);
      if (gid < G) v = *reinterpret_cast<const uint2*>(qn + gid * D + kp * 32 + tig * 8 + 4 * w);
      bq[2 * kp + w][0] = v.x;
      bq[2 * kp + w][1] = v.y;
    }
  }
  // Slots 0..c-1 from the arena and the new token (index c) from its own k
  // row, 16 per tile; tiles are dealt to the warps in turn.
  const int cnt = c + 1;
  const int ntiles = (cnt + 15) / 16;
  for (int t = warp; t < ntiles; t += kDecodeThreads / 32) {
    const int j0 = t * 16 + gid, j1 = j0 + 8;  // this lane's two slot rows
    uint4 X[KP], Y[KP];
#pragma unroll
    for (int kp = 0; kp < KP; ++kp) {
      const int off = kp * 32 + tig * 8;
      X[kp] = make_uint4(0, 0, 0, 0);
      Y[kp] = make_uint4(0, 0, 0, 0);
      if (j0 < c) X[kp] = __ldcs(reinterpret_cast<const uint4*>(Kb + static_cast<size_t>(j0) * D + off));
      else if (j0 == c) X[kp] = *reinterpret_cast<const uint4*>(kn + off);
      if (j1 < c) Y[kp] = __ldcs(reinterpret_cast<const uint4*>(Kb + static_cast<size_t>(j1) * D + off));
      else if (j1 == c) Y[kp] = *reinterpret_cast<const uint4*>(kn + off);
    }
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int kp = 0; kp < KP; ++kp) {
      const uint32_t a0[4] = {X[kp].x, Y[kp].x, X[kp].y, Y[kp].y};
      const uint32_t a1[4] = {X[kp].z, Y[kp].z, X[kp].w, Y[kp].w};
      mma_16816(acc, a0, bq[2 * kp][0], bq[2 * kp][1]);
      mma_16816(acc, a1, bq[2 * kp + 1][0], bq[2 * kp + 1][1]);
    }
    // acc: (slot j0, heads 2tig, 2tig+1) and (slot j1, same heads)
    const int h0 = 2 * tig;
    if (h0 < G) {
      if (j0 < cnt) lg[h0 * ld + j0] = acc[0] * p.scale_log2;
      if (j1 < cnt) lg[h0 * ld + j1] = acc[2] * p.scale_log2;
    }
    if (h0 + 1 < G) {
      if (j0 < cnt) lg[(h0 + 1) * ld + j0] = acc[1] * p.scale_log2;
      if (j1 < cnt) lg[(h0 + 1) * ld + j1] = acc[3] * p.scale_log2;
    }
  }
}

// H2O / TOVA unit.  lg: [G][cap + 1] floats of shared memory.
//
// Logits: a warp takes 16 slots at a time and forms S[16 slots][8 heads] =
// K Q^T on the tensor core (m16n8k16, heads past G are zero columns).  The
// dot product runs over d in a permuted order that lets every lane fill its
// A fragment from 16-byte loads of whole K rows: in the k-step pair kp, lane
// quadrant t (= lane % 4) holds dims kp*32 + t*8 + [0, 8) of its two slot
// rows; k-step 2kp + w takes elements 4w .. 4w + 3 of that slice (the low two
// as fragment columns 2t, 2t+1, the high two as 2t+8, 2t+9), and Q's B
// fragment is loaded in the same order.
template <int D, int G>
__device__ void attend_unit(const DecodeParams& p, const DecLayer& ly, const UnitRef& r, int n, int c,
                            float* lg, DecShared& sh) {
  const int ld = ly.cap + 1;  // row stride of lg
  const uint16_t* Kb = static_cast<const uint16_t*>(p.K) + r.rows0 * D;
  const uint16_t* kn = static_cast<const uint16_t*>(p.k_new[r.l]) + (static_cast<size_t>(r.s) * p.H_kv + r.h) * D;
  const uint16_t* qn = p.q_new[r.l] == nullptr
                           ? nullptr
                           : static_cast<const uint16_t*>(p.q_new[r.l]) +
                                 (static_cast<size_t>(r.s) * p.H_q + r.h * G) * D;

  // attention supplied by the caller's own decode attention: slots 0..c-1, then the new token
  const float* at = p.attn[r.l] == nullptr
                        ? nullptr
                        : p.attn[r.l] + (static_cast<size_t>(r.s) * p.H_kv + r.h) * static_cast<size_t>(ld);
  if (at == nullptr) unit_logits<D, G>(p, Kb, qn, kn, c, ld, lg);
  const int cnt = c + 1;
  __syncthreads();
  // per-head softmax statistics (not needed when the attention is supplied)
  float mg[G], zg[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    mg[g] = 0.f;
    zg[g] = 1.f;
  }
  if (at == nullptr) {
#pragma unroll
    for (int g = 0; g < G; ++g) {
      mg[g] = -INFINITY;
      for (int j = threadIdx.x; j < cnt; j += blockDim.x) mg[g] = fmaxf(mg[g], lg[g * ld + j]);
    }
    block_reduce_heads<G, true>(mg, sh);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      zg[g] = 0.f;
      for (int j = threadIdx.x; j < cnt; j += blockDim.x) {  // each thread keeps its own exponentials
        const float e = exp2f(lg[g * ld + j] - mg[g]);
        lg[g * ld + j] = e;
        zg[g] += e;
      }
    }
    block_reduce_heads<G, false>(zg, sh);
#pragma unroll
    for (int g = 0; g < G; ++g) zg[g] = 1.0f / (static_cast<float>(G) * zg[g]);
  }
  // group-mean attention -> new keys (each thread overwrites row 0 at its own j only)
  const float* accr = p.acc + r.rows0;
  const int32_t* posr = p.pos + r.rows0;
  const int limit = n + 1 - ly.r;  // positions >= limit are protected
  float ba = INFINITY;
  int bp = -1, bs = -1;
  constexpr int kU = 4;  // slots per thread whose global loads are issued together
  for (int j0 = threadIdx.x; j0 < cnt; j0 += kU * kDecodeThreads) {
    float accv[kU], atv[kU];
    int posv[kU];
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int j = j0 + q * kDecodeThreads;
      accv[q] = (ly.method == KVEV_H2O && j < c) ? accr[j] : 0.f;
      posv[q] = j < c ? posr[j] : n;
      atv[q] = (at != nullptr && j < cnt) ? at[j] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int j = j0 + q * kDecodeThreads;
      if (j >= cnt) break;
      float pj = atv[q];
      if (at == nullptr) {  // group mean of the kept exponentials times 1 / (G z_g)
        pj = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) pj += lg[g * ld + j] * zg[g];
      }
      const float a = accv[q] + pj;
      lg[j] = a;
      const int pos = posv[q];
      if (pos >= 0 && pos < limit && (bp < 0 || evict_before(a, pos, ba, bp))) {
        ba = a;
        bp = pos;
        bs = j;
      }
    }
  }
  const bool full = c >= ly.b;
  const int ev = full ? block_evict_choice(ba, bp, bs, sh) : -1;  // c = the new token
  __syncthreads();
  const int evicted_pos = ev < 0 ? -1 : (ev < c ? posr[ev] : n);
  __syncthreads();  // every thread has read posr[ev] before it is overwritten
  for (int j = threadIdx.x; j < c; j += blockDim.x)
    if (j != ev) p.acc[r.rows0 + j] = lg[j];
  if (!full) {
    if (c >= ly.cap) {  // never for a consistent state: slots of an evicting layer stay <= b
      if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
      return;
    }
    place_new(p, r, D, c, n, lg[c], c + 1, -1);
  } else if (ev < 0) {  // no evictable slot (protected window covers the cache)
    if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
  } else {
    place_new(p, r, D, ev < c ? ev : -1, n, lg[c], c, evicted_pos);
  }
}

constexpr int kDecodeWarps = kDecodeThreads / 32;

// The first layer whose prefix end (att_end or cheap_end) exceeds i: the
// layer holding the i-th unit of that kind.
template <bool kAttend>
__device__ __forceinline__ int find_kind_layer(const DecodeParams& p, int i) {
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if ((kAttend ? p.layer[mid].att_end : p.layer[mid].cheap_end) > i) hi = mid;
    else lo = mid + 1;
  }
  return lo;
}

__device__ __forceinline__ UnitRef unit_ref(const DecodeParams& p, int l, int rem) {
  const DecLayer& ly = p.layer[l];
  UnitRef r;
  r.l = l;
  r.s = rem / p.H_kv;
  r.h = rem - r.s * p.H_kv;
  r.u = ly.unit_off + rem;
  r.rows0 = static_cast<size_t>(ly.row_off) + static_cast<size_t>(rem) * ly.cap;
  return r;
}

// The step of the a-th H2O / TOVA unit (called by the whole block; returns
// early on an inconsistent state, which it records in the status word).
template <int D, int G>
__device__ __forceinline__ void step_attend(const DecodeParams& p, int a, float* lg, DecShared& sh) {
  const int l = find_kind_layer<true>(p, a);
  const DecLayer& ly = p.layer[l];
  const UnitRef r = unit_ref(p, l, a - (ly.att_end - p.B * p.H_kv));
  const int n = p.lens[r.s];
  const int c = p.count[r.u];
  if (c < 0 || c > ly.cap) {
    if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
    return;
  }
  attend_unit<D, G>(p, ly, r, n, c, lg, sh);
}

// place_new by one warp: the new token's K/V row (16-byte vectors over the
// lanes), then its bookkeeping by lane 0.
__device__ __forceinline__ void place_new_warp(const DecodeParams& p, const UnitRef& r, int D, int dst, int n,
                                               float acc_new, int new_count, int evicted_pos) {
  const int lane = threadIdx.x & 31;
  if (dst >= 0) {
    const int vec = D / 8;
    const size_t src = static_cast<size_t>(r.s) * p.H_kv + r.h;
    for (int i = lane; i < 2 * vec; i += 32) {
      const bool isv = i >= vec;
      const int e = isv ? i - vec : i;
      uint4* drow = reinterpret_cast<uint4*>(isv ? p.V : p.K) + (r.rows0 + dst) * vec + e;
      const uint4* srow = reinterpret_cast<const uint4*>(isv ? p.v_new[r.l] : p.k_new[r.l]) + src * vec + e;
      *drow = *srow;
    }
  }
  if (lane == 0) {
    if (dst >= 0) {
      p.pos[r.rows0 + dst] = n;
      p.acc[r.rows0 + dst] = acc_new;
    }
    p.count[r.u] = new_count;
    p.evicted[r.u] = evicted_pos;
  }
}

// The step of the i-th StreamingLLM or append-only unit, by one warp (no
// block barrier): StreamingLLM evicts the smallest position >= sink once
// sink + recent slots are held; an append-only unit takes the next slot.
__device__ void step_cheap_warp(const DecodeParams& p, int i, int D) {
  const int lane = threadIdx.x & 31;
  const int l = find_kind_layer<false>(p, i);
  const DecLayer& ly = p.layer[l];
  const UnitRef r = unit_ref(p, l, i - (ly.cheap_end - p.B * p.H_kv));
  const int n = p.lens[r.s];
  const int c = p.count[r.u];
  const bool streaming = ly.method == KVEV_STREAMING;
  if (c < 0 || c > ly.cap || (!streaming && c >= ly.cap) ||
      (streaming && c + 1 <= ly.sink + ly.recent && c >= ly.cap)) {
    if (lane == 0) atomicOr(p.status, kStatusDevice);
    return;
  }
  if (!streaming || c + 1 <= ly.sink + ly.recent) {  // append
    place_new_warp(p, r, D, c, n, 0.f, c + 1, -1);
    return;
  }
  // smallest position >= sink among the slots and the new token (positions are distinct)
  int bp = 0x7FFFFFFF, bs = -1;
  for (int j = lane; j <= c; j += 32) {
    const int pos = j < c ? p.pos[r.rows0 + j] : n;
    if (pos >= ly.sink && pos < bp) {
      bp = pos;
      bs = j;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int bp2 = __shfl_xor_sync(0xffffffffu, bp, o);
    const int bs2 = __shfl_xor_sync(0xffffffffu, bs, o);
    if (bp2 < bp) {
      bp = bp2;
      bs = bs2;
    }
  }
  __syncwarp();  // every lane has read the positions before slot bs is rewritten
  if (bs < 0) {
    if (lane == 0) atomicOr(p.status, kStatusDevice);
    return;
  }
  place_new_warp(p, r, D, bs < c ? bs : -1, n, 0.f, c, bp);
}

template <int D, int G>
__global__ void __launch_bounds__(kDecodeThreads) decode_step_kernel(const __grid_constant__ DecodeParams p) {
  extern __shared__ float lg[];
  __shared__ DecShared sh;
  // CTAs [0, n_att): one H2O / TOVA unit each; then eight cheap units per CTA
  if (static_cast<int>(blockIdx.x) < p.n_att) {
    step_attend<D, G>(p, blockIdx.x, lg, sh);
  } else {
    const int i = (blockIdx.x - p.n_att) * kDecodeWarps + (threadIdx.x >> 5);
    if (i < p.n_cheap) step_cheap_warp(p, i, D);
  }
  // The last CTA of the step to finish advances every sequence by one token:
  // every other CTA has read lens before it counted itself done.
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(p.done, 1) == static_cast<int>(gridDim.x) - 1) {
      for (int s = 0; s < p.B; ++s) p.lens[s] += 1;
      *p.done = 0;
      __threadfence();
    }
  }
}

// A step of a route without decode units: the sequences are one token longer.
__global__ void decode_advance_kernel(int32_t* lens, int B) {
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < B; s += gridDim.x * blockDim.x) lens[s] += 1;
}

// Decode arena from the packed prefill output: slot j < kept count of unit
// (l, s, h) takes prefill row j (its position and, for H2O prefill layers,
// its score as the initial acc); the remaining slots are marked empty.
__global__ void __launch_bounds__(kDecodeThreads) decode_init_kernel(const __grid_constant__ DecodeParams p) {
  const int u = blockIdx.x;
  const int l = find_dec_layer(p, u);
  const DecLayer& ly = p.layer[l];
  const int rem = u - ly.unit_off;
  const size_t rows0 = static_cast<size_t>(ly.row_off) + static_cast<size_t>(rem) * ly.cap;
  const size_t pre0 = static_cast<size_t>(ly.pre_row_off) + static_cast<size_t>(rem) * ly.pre_slots;
  int c = p.pre_count[static_cast<size_t>(l) * p.B * p.H_kv + rem];
  if (c < 0 || c > ly.pre_slots) {
    if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
    c = 0;
  }
  const int vec = p.d / 8;  // 16-byte vectors per row
  for (int i = threadIdx.x; i < c * vec; i += blockDim.x) {
    const int j = i / vec, e = i - j * vec;
    reinterpret_cast<uint4*>(p.K)[(rows0 + j) * vec + e] = reinterpret_cast<const uint4*>(p.pre_K)[(pre0 + j) * vec + e];
    reinterpret_cast<uint4*>(p.V)[(rows0 + j) * vec + e] = reinterpret_cast<const uint4*>(p.pre_V)[(pre0 + j) * vec + e];
  }
  const bool seed_acc = ly.pre_method == KVEV_H2O && p.h2o_state != nullptr;
  for (int j = threadIdx.x; j < ly.cap; j += blockDim.x) {
    p.pos[rows0 + j] = j < c ? p.pre_idx[pre0 + j] : -1;
    p.acc[rows0 + j] = (j < c && seed_acc) ? p.h2o_state[pre0 + j] : 0.f;
  }
  if (threadIdx.x == 0) {
    p.count[u] = c;
    p.evicted[u] = -1;
    if (u == 0) *p.done = 0;
  }
  if (u == 0)  // the first unit also copies the sequence lengths
    for (int i = threadIdx.x; i < p.B; i += blockDim.x) p.lens[i] = p.lens_in[i];
}

template <int D, int G>
cudaError_t launch_step_dg(const DecodeParams& p, size_t smem, cudaStream_t st) {
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(decode_step_kernel<D, G>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  const int grid = p.n_att + (p.n_cheap + kDecodeWarps - 1) / kDecodeWarps;
  decode_step_kernel<D, G><<<grid, kDecodeThreads, smem, st>>>(p);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_step_d(const DecodeParams& p, size_t smem, cudaStream_t st) {
  switch (p.G) {
    case 1: return launch_step_dg<D, 1>(p, smem, st);
    case 2: return launch_step_dg<D, 2>(p, smem, st);
    case 4: return launch_step_dg<D, 4>(p, smem, st);
    case 8: return launch_step_dg<D, 8>(p, smem, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool decode_supported(int d, int G) {
  return (d == 64 || d == 128) && (G == 1 || G == 2 || G == 4 || G == 8);
}

cudaError_t launch_decode_init(const DecodeParams& p, cudaStream_t st) {
  if (p.units == 0) return cudaSuccess;
  decode_init_kernel<<<p.units, kDecodeThreads, 0, st>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_decode_step(const DecodeParams& p, size_t smem, cudaStream_t st) {
  if (p.units > 0)  // the step kernel advances lens itself
    return p.d == 64 ? launch_step_d<64>(p, smem, st) : launch_step_d<128>(p, smem, st);
  decode_advance_kernel<<<1, 256, 0, st>>>(p.lens, p.B);
  return cudaGetLastError();
}

}  // namespace kvev
