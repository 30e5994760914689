// h2o_full.cu -- H2O prefill scores over every prompt query row (the
// accumulated attention of H2O's own scoring, Sec. 2.1).  For a unit u = (H2O
// layer, sequence s, KV head h) with n prompt positions, group heads g < G and
// c = log2(e) / sqrt(d):
//
//   lse2[g][t] = log2 sum_{k <= t} exp2(c q_{g,t} . k_k)
//   raw[k]     = (1/G) sum_g sum_{t = k}^{n-1} exp2(c q_{g,t} . k_k - lse2[g][t])
//
// Two launches in the FlashAttention arrangement, with no CTA ever waiting on
// another:
//   row pass (phase 0): an item is (unit, block of Pb positions).  The block's
//     R = G*Pb query rows sit on TMEM lanes and sweep the keys [0, block end)
//     on the tensor core (S = Q K^T over 256-key super-tiles), keeping each
//     row's running max and sum of exp2; the four softmax warpgroups' partials
//     are merged into lse2 of every prompt row.
//   key pass (phase 1): an item is (unit, 256-key super-tile).  Its keys sit on
//     TMEM lanes and sweep the query blocks whose rows can see them (S^T =
//     K Q^T), summing exp2(s*c - lse2_r) over the rows in registers.  Each
//     key's score is written once, by the item that holds the key, so the
//     result does not depend on the schedule.
// Items are dealt round-robin over the CTAs, heaviest first: row blocks from
// the end of the prompt, key super-tiles from its start.
//
// Roles per CTA (640 threads): warp 0 issues the TMA loads (one thread), warp
// 1 owns TMEM and issues tcgen05.mma (one thread), warp 2 stages each query
// block's -lse2 for the key pass, warps 4-19 are four softmax warpgroups that
// split every 256-column TMEM unit by columns (64 each).
#include "score_common.cuh"

namespace kvev {

namespace {

constexpr int kStreamStages = 2;
constexpr int kBufRows = 256;  // rows of every operand buffer: a Q block (<= 256 rows) or a K super-tile

struct FSmem {
  uint8_t* fixed;  // the item's own operand: Q block (phase 0) or K super-tile (phase 1)
  uint8_t* stage;  // kStreamStages streamed operands: K super-tiles (0) or Q blocks (1)
  float* lam;      // [2][256] -lse2 of a query block's rows; -inf where the row does not exist
  int* tpos;       // [2][256] prompt position of each row of that block; -1: no such row
  float2* pc;      // [kSoftmaxWGs][256] (max, sum) of each row (phase 0); in phase 1 the
                   // floats [kSoftmaxWGs][2][128] hold the partial sums of the item's keys
  uint64_t* ffull;
  uint64_t* fempty;
  uint64_t* sfull;
  uint64_t* sempty;
  uint64_t* tfull;
  uint64_t* tempty;
  uint64_t* lfull;
  uint64_t* lempty;
  uint64_t* done;
  uint32_t* tmem_slot;
};

__host__ __device__ __forceinline__ size_t fsmem_size(int D, size_t* stage_off, size_t* lam_off,
                                                       size_t* tpos_off, size_t* pc_off, size_t* bar_off) {
  const size_t buf = static_cast<size_t>(kBufRows) * D * 2;
  size_t off = buf;
  *stage_off = off;
  off += kStreamStages * buf;
  *lam_off = off;
  off += sizeof(float) * 2 * 256;
  *tpos_off = off;
  off += sizeof(int) * 2 * 256;
  *pc_off = off;
  off += sizeof(float2) * kSoftmaxWGs * 256;
  *bar_off = off;
  off += sizeof(uint64_t) * (2 + 2 * kStreamStages + 2 * kSlots + 4 + 1);
  off += sizeof(uint32_t);
  return off;
}

__device__ __forceinline__ FSmem fcarve(uint8_t* base, int D) {
  FSmem s;
  size_t so, lo, to, po, bo;
  fsmem_size(D, &so, &lo, &to, &po, &bo);
  s.fixed = base;
  s.stage = base + so;
  s.lam = reinterpret_cast<float*>(base + lo);
  s.tpos = reinterpret_cast<int*>(base + to);
  s.pc = reinterpret_cast<float2*>(base + po);
  uint64_t* b = reinterpret_cast<uint64_t*>(base + bo);
  s.ffull = b;
  s.fempty = b + 1;
  s.sfull = b + 2;
  s.sempty = s.sfull + kStreamStages;
  s.tfull = s.sempty + kStreamStages;
  s.tempty = s.tfull + kSlots;
  s.lfull = s.tempty + kSlots;
  s.lempty = s.lfull + 2;
  s.done = s.lempty + 2;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.done + 1);
  return s;
}

// Item i of the pass.  Units are the H2O layers' (sequence, KV head) pairs;
// items run unit-fastest so that the items in flight together share the
// heaviest block index.  False if the item is empty (beyond its sequence).
struct FItem {
  int hu;    // H2O unit (index into the lse array)
  int u;     // scoring unit (index into the score array)
  int ls, s, h, n;
  int blk;   // query block (phase 0) or key super-tile (phase 1)
};

__device__ __forceinline__ bool fitem(const ScoreParams& p, int i, FItem& f) {
  const int per_layer = p.B * p.H_kv;
  const int nu = p.n_h2o * per_layer;
  const int r = i / nu;
  f.hu = i - r * nu;
  const int li = f.hu / per_layer;
  const int rem = f.hu - li * per_layer;
  f.ls = p.h2o_slot[li];
  f.s = rem / p.H_kv;
  f.h = rem - f.s * p.H_kv;
  f.u = f.ls * per_layer + rem;
  f.n = p.lens[f.s];
  if (p.phase == 0) {
    f.blk = p.nb_max - 1 - r;
    return f.blk * p.Pb < f.n;
  }
  f.blk = r;
  return f.blk * kSuperKeys < f.n;
}

// Streamed operands of an item: the key super-tiles up to the block's end
// (phase 0), or the query blocks from the one holding the item's first key to
// the last of the prompt (phase 1).
__device__ __forceinline__ int n_stream(const ScoreParams& p, const FItem& f) {
  if (p.phase == 0) return (min(f.n, (f.blk + 1) * p.Pb) + kSuperKeys - 1) / kSuperKeys;
  return (f.n + p.Pb - 1) / p.Pb - (f.blk * kSuperKeys) / p.Pb;
}

// 128-key halves of a key super-tile that hold keys of the prompt.
__device__ __forceinline__ int n_halves(const FItem& f) {
  return min(2, (f.n - f.blk * kSuperKeys + kTileKeys - 1) / kTileKeys);
}

// Position of row r of the query block starting at q0, or -1 if the row does
// not exist (r >= R or beyond the prompt).  Rows are head-major: r = g*Pb + i.
__device__ __forceinline__ int block_row_pos(const ScoreParams& p, int r, int q0, int n) {
  if (r >= p.R) return -1;
  const int t = q0 + r % p.Pb;
  return t < n ? t : -1;
}

// ---------------------------------------------------------------------------
// Producer (one thread).
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void f_producer(const ScoreParams& p, const FSmem& sm) {
  constexpr uint32_t kBufBytes = kBufRows * D * 2;
  const uint32_t qbytes = static_cast<uint32_t>(p.R) * D * 2;  // what a G x Pb query box brings
  uint32_t e = 0, st = 0, ph = 0, issued = 0;
  bool ok = true;
  for (int i = blockIdx.x; ok && i < p.n_items; i += gridDim.x) {
    FItem f;
    if (!fitem(p, i, f)) continue;
    const CUtensorMap* kmap = &p.kmap[f.ls];
    const CUtensorMap* qmap = &p.qmap[f.ls];
    const int krow0 = (f.s * p.H_kv + f.h) * p.S_cap;
    const int qhead = f.s * p.H_q + f.h * p.G;
    // the fixed buffer is free once the previous item's MMAs have completed
    if (!wait_bar(sm.fempty, (e & 1) ^ 1, p)) { ok = false; break; }
    if (p.phase == 0) {
      mbar_expect_tx(sm.ffull, qbytes);
#pragma unroll
      for (int kc = 0; kc < D / 64; ++kc)
        tma_load_3d(sm.fixed + kc * (kBufRows * 128), qmap, kc * 64, f.blk * p.Pb, qhead, sm.ffull);
    } else {
      mbar_expect_tx(sm.ffull, kBufBytes);
#pragma unroll
      for (int kc = 0; kc < D / 64; ++kc)
        tma_load_2d(sm.fixed + kc * (kBufRows * 128), kmap, kc * 64, krow0 + f.blk * kSuperKeys, sm.ffull);
    }
    ++e;
    const int ns = n_stream(p, f);
    const int qb0 = (f.blk * kSuperKeys) / p.Pb;
    for (int j = 0; j < ns; ++j) {
      if (!wait_bar(&sm.sempty[st], ph ^ 1, p)) { ok = false; break; }
      uint8_t* dst = sm.stage + static_cast<size_t>(st) * kBufBytes;
      if (p.phase == 0) {
        mbar_expect_tx(&sm.sfull[st], kBufBytes);
#pragma unroll
        for (int kc = 0; kc < D / 64; ++kc)
          tma_load_2d(dst + kc * (kBufRows * 128), kmap, kc * 64, krow0 + j * kSuperKeys, &sm.sfull[st]);
      } else {
        mbar_expect_tx(&sm.sfull[st], qbytes);
#pragma unroll
        for (int kc = 0; kc < D / 64; ++kc)
          tma_load_3d(dst + kc * (kBufRows * 128), qmap, kc * 64, (qb0 + j) * p.Pb, qhead, &sm.sfull[st]);
      }
      ++issued;
      if (++st == kStreamStages) { st = 0; ph ^= 1; }
    }
  }
  // After an abort, wait (bounded) for the copies still landing in shared
  // memory before the CTA retires.
  if (!ok) {
    if (e > 0) wait_bar_drain(sm.ffull, (e - 1) & 1, 100000000ull);
    for (uint32_t b = 0; b < kStreamStages && b < issued; ++b) {
      const uint32_t last = ((issued - 1 - b) / kStreamStages) * kStreamStages + b;
      wait_bar_drain(&sm.sfull[b], (last / kStreamStages) & 1, 100000000ull);
    }
  }
}

// ---------------------------------------------------------------------------
// MMA issuer (one warp, an elected lane issues).
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void f_mma(const ScoreParams& p, const FSmem& sm, uint32_t tmem_base) {
  constexpr uint32_t kBufBytes = kBufRows * D * 2;
  constexpr uint32_t kColStep = kBufRows * 128 / 16;  // descriptor step between 64-column blocks
  constexpr uint32_t kHalf = 128 * 128 / 16;          // rows (or keys) 128..255 of a buffer
  // phase 0: S[128 rows of a group][256 keys]; phase 1: S^T[128 keys of a half][R_pad rows]
  const uint32_t idesc = p.phase == 0 ? idesc_bf16_f32(128, kSuperKeys) : idesc_bf16_f32(128, p.R_pad);
  const int groups = p.R_pad > 128 ? 2 : 1;
  uint32_t e = 0, st = 0, kph = 0, sl = 0, tph = 0;
  bool ok = true;
  for (int i = blockIdx.x; ok && i < p.n_items; i += gridDim.x) {
    FItem f;
    if (!fitem(p, i, f)) continue;
    if (!wait_bar_warp(sm.ffull, e & 1, p)) { ok = false; break; }
    tc_fence_after();
    const uint64_t fdesc = sw128_desc(smem_u32(sm.fixed));
    const int ns = n_stream(p, f);
    const int nu = p.phase == 0 ? groups : n_halves(f);
    for (int j = 0; ok && j < ns; ++j) {
      if (!wait_bar_warp(&sm.sfull[st], kph, p)) { ok = false; break; }
      tc_fence_after();
      const uint64_t sdesc = sw128_desc(smem_u32(sm.stage) + st * kBufBytes);
      for (int u = 0; u < nu; ++u) {
        if (!wait_bar_warp(&sm.tempty[sl], tph ^ 1, p)) { ok = false; break; }
        tc_fence_after();
        const uint32_t dcol = tmem_base + sl * kSlotCols;
        // A = the fixed buffer's rows 128u.. (phase 0: row group u of the Q
        // block; phase 1: key half u of the K super-tile), B = the streamed
        // buffer (phase 0: 256 keys; phase 1: the block's R_pad rows)
        const uint64_t adesc = fdesc + static_cast<uint64_t>(u * kHalf);
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
          const uint32_t off = (k >> 2) * kColStep + (k & 3) * 2;
          umma_bf16_elect(dcol, adesc + off, sdesc + off, idesc, k > 0);
        }
        umma_commit_elect(&sm.tfull[sl]);
        sl += 2;
        if (sl == kSlots) { sl = 0; tph ^= 1; }
      }
      if (!ok) break;
      umma_commit_elect(&sm.sempty[st]);
      if (++st == kStreamStages) { st = 0; kph ^= 1; }
    }
    if (!ok) break;
    umma_commit_elect(sm.fempty);  // the fixed buffer is free once these MMAs finish
    ++e;
  }
  umma_commit_elect(sm.done);
  wait_bar_drain(sm.done, 0, 1000000000ull);
}

// ---------------------------------------------------------------------------
// Normaliser stager (phase 1, one warp): -lse2 and the position of every row
// of each query block, in the order the softmax warpgroups consume them.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void f_lam(const ScoreParams& p, const FSmem& sm) {
  const int lane = threadIdx.x & 31;
  uint32_t lq = 0;
  for (int i = blockIdx.x; i < p.n_items; i += gridDim.x) {
    FItem f;
    if (!fitem(p, i, f)) continue;
    const int qb0 = (f.blk * kSuperKeys) / p.Pb;
    const int ns = n_stream(p, f);
    const float* lse = p.lse + static_cast<size_t>(f.hu) * p.G * p.S_cap;
    // lane's eight rows of a block: position (or -1) and lse2, all loads in
    // flight at once; block j + 1's loads go out before the wait for its buffer
    float v[8];
    int tt[8];
    auto fetch = [&](int j) {
      const int q0 = (qb0 + j) * p.Pb;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int r = lane + 32 * q;
        tt[q] = block_row_pos(p, r, q0, f.n);
        v[q] = tt[q] >= 0 ? __ldcg(&lse[static_cast<size_t>(r / p.Pb) * p.S_cap + tt[q]]) : INFINITY;
      }
    };
    fetch(0);
    for (int j = 0; j < ns; ++j) {
      const uint32_t lb = lq & 1;
      if (!wait_bar_warp(&sm.lempty[lb], ((lq >> 1) & 1) ^ 1, p)) return;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        sm.lam[lb * 256 + lane + 32 * q] = -v[q];
        sm.tpos[lb * 256 + lane + 32 * q] = tt[q];
      }
      __syncwarp();
      mbar_arrive_elect(&sm.lfull[lb]);
      ++lq;
      if (j + 1 < ns) fetch(j + 1);
    }
  }
}

// ---------------------------------------------------------------------------
// Softmax warpgroups.
// ---------------------------------------------------------------------------

// This warpgroup's 64 columns of a 256-column unit, released before use.
__device__ __forceinline__ void f_take(const FSmem& sm, uint32_t lane_base, uint32_t g, uint32_t (&r0)[32],
                                       uint32_t (&r1)[32]) {
  const uint32_t s0 = g & (kSlots - 1);
  tmem_ld64_async(lane_base + s0 * kSlotCols, r0, r1);
  tmem_wait64(r0, r1);
  tc_fence_before();
  __syncwarp();
  mbar_arrive_elect(&sm.tempty[s0]);
}

__device__ __forceinline__ int lds1i(const int* p) {
  int v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)));
  return v;
}

// Key sum over 32 rows with per-row checks: rows that do not exist (tp < 0)
// or that cannot see key k (k > position) add nothing.
__device__ __forceinline__ void s2_chunk_rows(const uint32_t (&rr)[32], float c, const float* nl, const int* tp,
                                              int k, float2 (&a)[4]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    if (k <= lds1i(tp + i)) {
      const float e = ex2_approx(fmaf(__uint_as_float(rr[i]), c, lds1(nl + i)));
      if (i & 1) a[(i >> 1) & 3].y += e; else a[(i >> 1) & 3].x += e;
    }
  }
}

__device__ __forceinline__ void f_softmax(const ScoreParams& p, const FSmem& sm, uint32_t tmem_base, int wg) {
  const int warp = threadIdx.x >> 5;
  const int quarter = warp & 3;
  const int lrow = quarter * 32 + (threadIdx.x & 31);  // TMEM lane: row (phase 0) / key (phase 1)
  const int stid = threadIdx.x - 128;                  // 0..511 over the softmax warpgroups
  const uint32_t lane_base =
      tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(64 * wg);
  const int groups = p.R_pad > 128 ? 2 : 1;
  const float c = p.scale_log2;
  float* red = reinterpret_cast<float*>(sm.pc);
  uint32_t g = 0, lq = 0;
  bool ok = true;
  for (int i = blockIdx.x; i < p.n_items; i += gridDim.x) {
    FItem f;
    if (!fitem(p, i, f)) continue;
    const int ns = n_stream(p, f);
    if (p.phase == 0) {
      // ---- rows: running (max, sum) of exp2 over the block's prefix keys ----
      const int q0 = f.blk * p.Pb;
      const int tr0 = block_row_pos(p, lrow, q0, f.n);
      const int tr1 = block_row_pos(p, 128 + lrow, q0, f.n);
      float m0 = -INFINITY, z0 = 0.f, m1 = -INFINITY, z1 = 0.f;
      for (int j = 0; j < ns; ++j) {
        const int kb = j * kSuperKeys;
        const int k0 = kb + 64 * wg;                  // this warpgroup's keys k0 .. k0 + 63
        const bool full = kb + kSuperKeys - 1 <= q0;  // every key visible to every row of the block
        for (int hh = 0; hh < groups; ++hh) {
          if (ok && !wait_bar(&sm.tfull[g & (kSlots - 1)], (g / kSlots) & 1, p)) ok = false;
          uint32_t r0[32], r1[32];
          f_take(sm, lane_base, g, r0, r1);
          float v0[32], v1[32];
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            v0[q] = __uint_as_float(r0[q]);
            v1[q] = __uint_as_float(r1[q]);
          }
          const int tr = hh == 0 ? tr0 : tr1;
          if (!full) {
            mask_chunk(v0, k0, tr);
            mask_chunk(v1, k0 + 32, tr);
          }
          if (hh == 0)
            s1_chunk64(v0, v1, c, m0, z0);
          else
            s1_chunk64(v0, v1, c, m1, z1);
          g += 2;
        }
      }
      sm.pc[wg * 256 + lrow] = make_float2(m0, z0);
      if (groups == 2) sm.pc[wg * 256 + 128 + lrow] = make_float2(m1, z1);
      named_bar_sync(1, 128 * kSoftmaxWGs);
      float* lse = p.lse + static_cast<size_t>(f.hu) * p.G * p.S_cap;
      for (int r = stid; r < p.R; r += 128 * kSoftmaxWGs) {
        const int t = block_row_pos(p, r, q0, f.n);
        float2 a = sm.pc[r];
#pragma unroll
        for (int w = 1; w < kSoftmaxWGs; ++w) a = merge_ms(a, sm.pc[w * 256 + r]);
        if (ok && t >= 0)
          lse[static_cast<size_t>(r / p.Pb) * p.S_cap + t] =
              (a.x == -INFINITY || a.y <= 0.f) ? INFINITY : a.x + lg2_approx(a.y);
      }
      named_bar_sync(1, 128 * kSoftmaxWGs);
    } else {
      // ---- keys: sum of exp2(s*c - lse2) over every row that sees the key ----
      const int key0 = f.blk * kSuperKeys;
      const int halves = n_halves(f);
      const int qb0 = key0 / p.Pb;
      float2 a[2][4];
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int q = 0; q < 4; ++q) a[hh][q] = make_float2(0.f, 0.f);
      const int ra0 = 64 * wg, rb0 = 64 * wg + 32;  // this warpgroup's rows of the block
      for (int j = 0; j < ns; ++j) {
        const uint32_t lb = lq & 1;
        if (ok && !wait_bar(&sm.lfull[lb], (lq >> 1) & 1, p)) ok = false;
        const float* nl = sm.lam + lb * 256;
        const int* tp = sm.tpos + lb * 256;
        const int q0 = (qb0 + j) * p.Pb;
        // no causal cut inside this block and every one of its rows exists
        const bool clear = key0 + kSuperKeys - 1 <= q0 && q0 + p.Pb <= f.n;
        for (int hh = 0; hh < halves; ++hh) {
          if (ok && !wait_bar(&sm.tfull[g & (kSlots - 1)], (g / kSlots) & 1, p)) ok = false;
          uint32_t ra[32], rb[32];
          f_take(sm, lane_base, g, ra, rb);
          const int k = key0 + kTileKeys * hh + lrow;
          if (ok) {
            if (clear && ra0 + 32 <= p.R)
              s2_chunk_full(ra, c, nl + ra0, a[hh]);
            else if (ra0 < p.R_pad)
              s2_chunk_rows(ra, c, nl + ra0, tp + ra0, k, a[hh]);
            if (clear && rb0 + 32 <= p.R)
              s2_chunk_full(rb, c, nl + rb0, a[hh]);
            else if (rb0 < p.R_pad)
              s2_chunk_rows(rb, c, nl + rb0, tp + rb0, k, a[hh]);
          }
          g += 2;
        }
        __syncwarp();
        mbar_arrive_elect(&sm.lempty[lb]);
        ++lq;
      }
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
        if (hh < halves) red[(wg * 2 + hh) * 128 + lrow] = sum4x2(a[hh]);
      named_bar_sync(1, 128 * kSoftmaxWGs);
      float* out = p.raw + static_cast<size_t>(f.u) * p.S_cap;
      for (int q = stid; q < halves * 128; q += 128 * kSoftmaxWGs) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kSoftmaxWGs; ++w) sum += red[(w * 2 + q / 128) * 128 + (q & 127)];
        if (ok && key0 + q < f.n) out[key0 + q] = sum * p.inv_G;
      }
      named_bar_sync(1, 128 * kSoftmaxWGs);
    }
  }
}

template <int D>
__global__ void __launch_bounds__(kScoreThreads, 1) h2o_full_kernel(const __grid_constant__ ScoreParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {  // the 128-byte swizzle needs 1024-byte aligned buffers
    if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
    return;
  }
  const FSmem sm = fcarve(smem_raw, D);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    mbar_init(sm.ffull, 1);
    mbar_init(sm.fempty, 1);
    for (int i = 0; i < kStreamStages; ++i) {
      mbar_init(&sm.sfull[i], 1);
      mbar_init(&sm.sempty[i], 1);
    }
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&sm.tfull[i], 1);
      mbar_init(&sm.tempty[i], 4 * kSoftmaxWGs);  // every softmax warp copies its slice
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.lfull[i], 1);
      mbar_init(&sm.lempty[i], 4 * kSoftmaxWGs);
    }
    mbar_init(sm.done, 1);
    fence_barrier_init();
    fence_proxy_async();
  }
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, kSlots * kSlotCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  if (warp < 4) {
    regs_dealloc<kRegsControl>();
    if (warp == 0 && (threadIdx.x & 31) == 0) f_producer<D>(p, sm);
    if (warp == 1) f_mma<D>(p, sm, tmem_base);
    if (warp == 2 && p.phase == 1) f_lam(p, sm);
  } else {
    regs_alloc<kRegsSoftmax>();
    f_softmax(p, sm, tmem_base, (warp - 4) >> 2);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kSlots * kSlotCols);
  }
}

// The caller's log-sum-exp of every prompt row (the softmax_lse its own
// prefill attention returns, natural log, fp32 [B][H_q][S_cap]) into the key
// pass's base-2 rows, in place of the row pass.  One CTA per H2O unit.
__global__ void __launch_bounds__(256) lse_rows_fill_kernel(const __grid_constant__ ScoreParams p) {
  const int per_layer = p.B * p.H_kv;
  const int hu = blockIdx.x;
  const int li = hu / per_layer;
  const int rem = hu - li * per_layer;
  const int s = rem / p.H_kv, h = rem - s * p.H_kv;
  const int n = p.lens[s];
  const float* src = p.lse_src[li] + (static_cast<size_t>(s) * p.H_q + static_cast<size_t>(h) * p.G) * p.S_cap;
  float* dst = p.lse + static_cast<size_t>(hu) * p.G * p.S_cap;
  constexpr float kInvLn2 = 1.4426950408889634f;
  for (int g = 0; g < p.G; ++g)
    for (int t = threadIdx.x; t < n; t += blockDim.x)
      dst[static_cast<size_t>(g) * p.S_cap + t] = __ldg(src + static_cast<size_t>(g) * p.S_cap + t) * kInvLn2;
}

}  // namespace

int h2o_full_smem_bytes(int d) {
  size_t so, lo, to, po, bo;
  const size_t off = fsmem_size(d, &so, &lo, &to, &po, &bo);
  return static_cast<int>((off + 127) & ~size_t(127));
}

int h2o_full_kernel_regs(int d) {
  cudaFuncAttributes a = {};
  const cudaError_t e = d == 64 ? cudaFuncGetAttributes(&a, h2o_full_kernel<64>)
                                : cudaFuncGetAttributes(&a, h2o_full_kernel<128>);
  return e == cudaSuccess ? a.numRegs : -1;
}

cudaError_t h2o_full_set_smem(int d, size_t smem) {
  if (d == 64)
    return cudaFuncSetAttribute(h2o_full_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem));
  return cudaFuncSetAttribute(h2o_full_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

cudaError_t launch_lse_rows_fill(const ScoreParams& p, cudaStream_t s) {
  const int units = p.n_h2o * p.B * p.H_kv;
  if (units == 0) return cudaSuccess;
  lse_rows_fill_kernel<<<units, 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_h2o_full(const ScoreParams& p, int d, int grid, size_t smem, cudaStream_t s) {
  if (grid <= 0) return cudaSuccess;
  if (d == 64)
    h2o_full_kernel<64><<<grid, kScoreThreads, smem, s>>>(p);
  else
    h2o_full_kernel<128><<<grid, kScoreThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvev
