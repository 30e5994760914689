// score.cu -- observation-window attention scores of every SnapKV / H2O layer
// (the scoring step of the rules Sec. 2.1 cites), for all layers of a route in
// one persistent, cooperative launch.
//
// For a unit u = (scoring layer, sequence s, KV head h) with n valid keys and
// the R = G*W window query rows of the group (row r = g*W + i sits at absolute
// position t_r = n - W + i and sees keys 0..t_r):
//
//   raw[k] = (1/G) * sum_r exp(q_r . k_k / sqrt(d) - lse_r)      (k <= t_r)
//   lse_r  = log sum_{k' <= t_r} exp(q_r . k_k' / sqrt(d))
//
// The row normaliser lse_r needs every key before any score is final, so the
// keys are swept twice:
//   sweep 1: S = Q K^T on the tensor core (rows on TMEM lanes), per-row running
//            max / sum of exp2 in registers -> per-chunk partials;
//   sweep 2: S^T = K Q^T on the tensor core (keys on TMEM lanes), each thread
//            owns one key and sums exp2(s*log2e/sqrt(d) - lse2_r) over the rows.
// Work items are chunks of chunk_keys keys.  A CTA runs sweep 1 of item j+1
// before sweep 2 of item j, so the re-read of item j's K tiles (one round of
// the whole grid later, ~grid*chunk bytes of new traffic) is served by L2 and
// the per-unit normaliser is ready without any CTA idling.  The last chunk of a
// unit to finish sweep 1 combines the partials and publishes lse (release
// flag); sweep-2 readers spin on it with a time bound.  All CTAs are
// co-resident (cooperative launch) and a unit spans at most two rounds of
// items, so the wait always ends.
//
// Roles per CTA (640 threads, five warpgroups): warp 0 issues TMA loads (one
// thread), warp 1 owns TMEM and issues tcgen05.mma (one thread), warps 2-3
// idle; warpgroups 1-4 are softmax warpgroups.  TMEM is four 128-column
// slots, one per 128-row group of a tile's accumulator (a tile uses one or
// two), and softmax warpgroup w owns slot w: it copies the slot to registers
// in 64-column pieces and releases it before the last piece's arithmetic, so
// the tensor core keeps filling the other slots meanwhile.  The softmax
// warpgroups never wait on each other.  setmaxnreg moves registers from
// warpgroup 0 to the softmax warpgroups.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

struct Smem {
  uint8_t* qbuf;     // two Q buffers of qbytes each, indexed arithmetically (a dynamically
  uint32_t qbytes;   // indexed member array would push the whole struct to local memory)
  uint8_t* kbuf;     // stages * tile bytes
  float* lam;        // [4][R_pad]: per-warpgroup copy of -lse2 of the current sweep-2 unit
  uint64_t* kfull;
  uint64_t* kempty;
  uint64_t* qfull;
  uint64_t* qempty;
  uint64_t* tfull;
  uint64_t* tempty;
  uint64_t* done;
  uint32_t* tmem_slot;
  int* flag;         // [8]: [wg] last-arrival of sweep 1, [4+wg] ready of sweep 2
};

__device__ __forceinline__ Smem carve(uint8_t* base, const ScoreParams& p, int D) {
  Smem s;
  size_t off = 0;
  const size_t qbytes = static_cast<size_t>(p.q_rows) * D * 2;
  const size_t tbytes = static_cast<size_t>(kTileKeys) * D * 2;
  s.qbuf = base + off;
  s.qbytes = static_cast<uint32_t>(qbytes);
  off += 2 * qbytes;
  s.kbuf = base + off;
  off += tbytes * p.stages;
  s.lam = reinterpret_cast<float*>(base + off);
  off += kSoftmaxWGs * sizeof(float) * p.R_pad;
  off = (off + 7) & ~size_t(7);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + off);
  s.kfull = bars;
  s.kempty = bars + p.stages;
  s.qfull = bars + 2 * p.stages;
  s.qempty = s.qfull + 2;
  s.tfull = s.qempty + 2;
  s.tempty = s.tfull + kSlots;
  s.done = s.tempty + kSlots;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.done + 1);
  s.flag = reinterpret_cast<int*>(s.tmem_slot + 1);
  return s;
}

struct ItemInfo {
  int u, s, h, ls, n, key0, ntiles, cs, nchunks;
};

// Work item t from its packed record (written by the prologue: one 16-byte load).
__device__ __forceinline__ int4 load_item(const ScoreParams& p, int t) { return __ldg(&p.item[t]); }

__device__ __forceinline__ ItemInfo decode_item(const ScoreParams& p, int t, int4 r) {
  ItemInfo it;
  it.u = r.x;
  it.n = r.y;
  it.key0 = r.z;
  it.ntiles = r.w & 0xFFFF;
  it.nchunks = r.w >> 16;
  it.cs = t - it.key0 / p.chunk_keys;
  const int per_layer = p.B * p.H_kv;
  it.ls = it.u / per_layer;
  const int rem = it.u - it.ls * per_layer;
  it.s = rem / p.H_kv;
  it.h = rem - it.s * p.H_kv;
  return it;
}

// Items a role needs at step j of the lag-1 loop: j (sweep 1) and j-1
// (sweep 2).  At step j it pulls the record of item j+1 into L1, so the load at
// step j+1 is an L1 hit instead of a round trip to L2 on the critical path.
__device__ __forceinline__ void prefetch_item(const ScoreParams& p, int first, int stride, int j, int J) {
  if (j + 1 < J) asm volatile("prefetch.global.L1 [%0];" ::"l"(p.item + first + (j + 1) * stride));
}

// Bounded wait on an mbarrier phase; false if it ran out or another role
// aborted.  Each try sleeps in hardware for up to kWaitSliceNs, so the abort
// flag and the time limit are checked at least that often.
constexpr uint32_t kWaitSliceNs = 20000;
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, const ScoreParams& p) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_sleep(bar, parity, kWaitSliceNs)) {
    if (ld_volatile(p.abort_flag)) return false;
    if (globaltimer_ns() - t0 > static_cast<uint64_t>(p.wait_ns)) {
      atomicExch(p.abort_flag, 1);
      atomicOr(p.status, kStatusTimeout);
      return false;
    }
  }
  return true;
}

// wait_bar by every lane of a warp; the warp agrees on the outcome (all lanes
// see the same phase eventually, but a time-out may hit only some of them).
__device__ __forceinline__ bool wait_bar_warp(uint64_t* bar, uint32_t parity, const ScoreParams& p) {
  return __all_sync(0xffffffffu, wait_bar(bar, parity, p));
}

// Bounded wait used while shutting down: ignores the abort flag, gives up after
// `ns` nanoseconds (asynchronous copies and MMAs finish on their own).
__device__ __forceinline__ void wait_bar_drain(uint64_t* bar, uint32_t parity, uint64_t ns) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_sleep(bar, parity, kWaitSliceNs))
    if (globaltimer_ns() - t0 > ns) return;
}

// ---------------------------------------------------------------------------
// Producer: TMA loads of Q (once per item) and of K tiles (twice per item).
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void producer(const ScoreParams& p, const Smem& sm, int first, int stride, int J) {
  constexpr uint32_t kTileBytes = kTileKeys * D * 2;
  const uint32_t qbytes = static_cast<uint32_t>(p.R_pad) * D * 2;
  const uint64_t keep = policy_evict_last();   // first read of a K tile: keep it for the re-read
  const uint64_t drop = policy_evict_first();  // second read: its last use
  uint32_t tile = 0;            // tiles issued (for the drain after an abort)
  uint32_t pst = 0, pph = 0;    // K stage ring: position and phase of the next tile
  int last_q_item = -1;
  int issued_q0 = 0, issued_q1 = 0;  // Q loads issued into each buffer
  bool ok = true;
  for (int j = 0; j <= J && ok; ++j) {
    prefetch_item(p, first, stride, j, J);
    for (int sweep = 0; sweep < 2 && ok; ++sweep) {
      const int jj = sweep == 0 ? j : j - 1;
      if (sweep == 0 && j >= J) continue;
      if (sweep == 1 && j == 0) continue;
      const int t = first + jj * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      const CUtensorMap* kmap = &p.kmap[it.ls];
      if (sweep == 0) {
        const int qb = jj & 1;
        if (!wait_bar(&sm.qempty[qb], ((jj >> 1) & 1) ^ 1, p)) { ok = false; break; }
        mbar_expect_tx(&sm.qfull[qb], qbytes);
        const int qrow = (it.s * p.H_q + it.h * p.G) * p.W;
#pragma unroll
        for (int kc = 0; kc < D / 64; ++kc)
          tma_load_2d(sm.qbuf + qb * sm.qbytes + static_cast<size_t>(kc) * p.q_rows * 128, &p.qmap[it.ls],
                      kc * 64, qrow, &sm.qfull[qb]);
        if (qb == 0) issued_q0 = jj + 1; else issued_q1 = jj + 1;
        last_q_item = jj;
      }
      const int row0 = (it.s * p.H_kv + it.h) * p.S_cap + it.key0;
      for (int i = 0; i < it.ntiles; ++i, ++tile) {
        const uint32_t st = pst, ph = pph;
        if (++pst == static_cast<uint32_t>(p.stages)) { pst = 0; pph ^= 1; }
        if (!wait_bar(&sm.kempty[st], ph ^ 1, p)) { ok = false; break; }
        uint8_t* dst = sm.kbuf + static_cast<size_t>(st) * kTileBytes;
        mbar_expect_tx(&sm.kfull[st], kTileBytes);
#pragma unroll
        for (int kc = 0; kc < D / 64; ++kc)
          tma_load_2d_hint(dst + kc * (kTileKeys * 128), kmap, kc * 64, row0 + i * kTileKeys,
                           &sm.kfull[st], sweep == 0 ? keep : drop);
      }
    }
  }
  (void)last_q_item;
  // Drain: make sure no copy is still landing in shared memory when the CTA
  // retires (only relevant after an abort; normally every load was consumed).
  if (!ok) {
    const uint32_t S = p.stages;
    for (uint32_t st = 0; st < S && st < tile; ++st) {
      const uint32_t last = ((tile - 1 - st) / S) * S + st;  // last tile issued into st
      wait_bar_drain(&sm.kfull[st], (last / S) & 1, 100000000ull);
    }
    if (issued_q0 > 0) wait_bar_drain(&sm.qfull[0], ((issued_q0 - 1) >> 1) & 1, 100000000ull);
    if (issued_q1 > 0) wait_bar_drain(&sm.qfull[1], ((issued_q1 - 1) >> 1) & 1, 100000000ull);
  }
}

// ---------------------------------------------------------------------------
// MMA issuer (one warp; an elected lane issues): sweep 1 -> S = Q K^T,
// sweep 2 -> S^T = K Q^T.
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void mma_issuer(const ScoreParams& p, const Smem& sm, uint32_t tmem_base, int first,
                           int stride, int J) {
  constexpr uint32_t kTileBytes = kTileKeys * D * 2;
  const int nh = p.R_pad > 128 ? 2 : 1;
  const uint32_t idesc1 = idesc_bf16_f32(128, kTileKeys);
  // sweep 2: N = rows of the group (128, or what is left of R_pad in the last group)
  const uint32_t idesc2a = idesc_bf16_f32(128, p.R_pad > 128 ? 128 : p.R_pad);
  const uint32_t idesc2b = idesc_bf16_f32(128, p.R_pad > 128 ? p.R_pad - 128 : 128);
  // descriptor steps (address / 16) between the 64-wide column blocks of Q and of a K tile
  const uint32_t qcol_step = static_cast<uint32_t>(p.q_rows) * 128 / 16;
  constexpr uint32_t kcol_step = kTileKeys * 128 / 16;
  uint32_t st = 0, kph = 0;  // K stage ring: position and phase of the next tile
  uint32_t sl = 0, tph = 0;  // TMEM slot ring: position and phase of the next slot
  bool ok = true;
  for (int j = 0; j <= J && ok; ++j) {
    prefetch_item(p, first, stride, j, J);
    for (int sweep = 0; sweep < 2 && ok; ++sweep) {
      const int jj = sweep == 0 ? j : j - 1;
      if (sweep == 0 && j >= J) continue;
      if (sweep == 1 && j == 0) continue;
      const int t = first + jj * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      const int qb = jj & 1;
      const uint64_t qdesc0 = sw128_desc(smem_u32(sm.qbuf) + qb * sm.qbytes);
      if (sweep == 0 && !wait_bar_warp(&sm.qfull[qb], (jj >> 1) & 1, p)) { ok = false; break; }
      const bool s1 = sweep == 0;
      const uint32_t astep = s1 ? qcol_step : kcol_step, bstep = s1 ? kcol_step : qcol_step;
      for (int i = 0; i < it.ntiles; ++i) {
        if (!wait_bar_warp(&sm.kfull[st], kph, p)) { ok = false; break; }
        // Descriptors of the tile and of the Q row group, built once: a
        // descriptor's low field is the address / 16, so the k-step offsets
        // (all inside shared memory, no carry out of the field) are plain adds.
        const uint64_t kdesc = sw128_desc(smem_u32(sm.kbuf) + st * kTileBytes);
        // One 128-column TMEM slot per 128-row group of Q: sweep 1 writes
        // S[rows of group h][keys], sweep 2 writes S^T[keys][rows of group h].
        for (int h = 0; h < nh; ++h) {
          if (!wait_bar_warp(&sm.tempty[sl], tph ^ 1, p)) { ok = false; break; }
          tc_fence_after();
          const uint32_t dcol = tmem_base + sl * kSlotCols;
          const uint64_t qdesc = qdesc0 + static_cast<uint64_t>(h * (128 * 128 / 16));
          const uint32_t idesc = s1 ? idesc1 : (h == 0 ? idesc2a : idesc2b);
          const uint64_t adesc = s1 ? qdesc : kdesc, bdesc = s1 ? kdesc : qdesc;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint32_t a = (k >> 2) * astep + (k & 3) * 2, b = (k >> 2) * bstep + (k & 3) * 2;
            umma_bf16_elect(dcol, adesc + a, bdesc + b, idesc, k > 0);
          }
          umma_commit_elect(&sm.tfull[sl]);
          if (++sl == kSlots) { sl = 0; tph ^= 1; }
        }
        if (!ok) break;
        umma_commit_elect(&sm.kempty[st]);
        if (++st == static_cast<uint32_t>(p.stages)) { st = 0; kph ^= 1; }
      }
      if (ok && sweep == 1) umma_commit_elect(&sm.qempty[qb]);
    }
  }
  // Every MMA issued so far has completed once `done` flips.
  umma_commit_elect(sm.done);
  wait_bar_drain(sm.done, 0, 1000000000ull);
}

// ---------------------------------------------------------------------------
// Softmax warpgroups.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int row_pos(const ScoreParams& p, int r, int n) {
  // absolute position of window row r; < 0 means the row lies before the sequence
  return n - p.W + (r % p.W);
}

__device__ __forceinline__ float max32(const float (&v)[32]) {
  float t[11];
#pragma unroll
  for (int j = 0; j < 10; ++j) t[j] = fmax3(v[3 * j], v[3 * j + 1], v[3 * j + 2]);
  t[10] = fmaxf(v[30], v[31]);
  const float a = fmax3(t[0], t[1], t[2]), b = fmax3(t[3], t[4], t[5]);
  const float c = fmax3(t[6], t[7], t[8]), e = fmax3(t[9], t[10], a);
  return fmax3(b, c, e);
}

__device__ __forceinline__ float sum8(const float (&a)[8]) {
  return ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
}

// One 32-key chunk of sweep 1 for one row: online base-2 (max, sum) update.
__device__ __forceinline__ void s1_chunk(const uint32_t (&rr)[32], float c, bool full, int k0,
                                         int tr, float& m, float& z) {
  float v[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(rr[i]);
  if (!full) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (k0 + i > tr) v[i] = -INFINITY;
  }
  const float mx = max32(v);
  if (mx == -INFINITY) return;
  const float mnew = fmaxf(m, mx * c);
  const float zs = z * ex2_approx(m - mnew);  // m = -inf -> 0
  const float2 cc = make_float2(c, c), nm = make_float2(-mnew, -mnew);
  float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 32; i += 2) {
    const float2 t = ffma2(make_float2(v[i], v[i + 1]), cc, nm);
    a[i & 7] += ex2_approx(t.x);
    a[(i + 1) & 7] += ex2_approx(t.y);
  }
  z = zs + sum8(a);
  m = mnew;
}

// One 32-row chunk of sweep 2 for this thread's key: sum of exp2(s*c - lse2_r)
// into eight accumulators; nl = -lse2 of the chunk's rows (shared memory).
__device__ __forceinline__ void s2_chunk(const ScoreParams& p, const uint32_t (&rr)[32], bool full,
                                         const float* nl, int r0, int k, int n, float (&a)[8]) {
  const float c = p.scale_log2;
  const float2 cc = make_float2(c, c);
  if (full) {
#pragma unroll
    for (int i = 0; i < 32; i += 4) {
      const float4 l4 = lds4(nl + i);
      const float2 t0 = ffma2(make_float2(__uint_as_float(rr[i]), __uint_as_float(rr[i + 1])), cc,
                              make_float2(l4.x, l4.y));
      const float2 t1 = ffma2(make_float2(__uint_as_float(rr[i + 2]), __uint_as_float(rr[i + 3])),
                              cc, make_float2(l4.z, l4.w));
      a[i & 7] += ex2_approx(t0.x);
      a[(i + 1) & 7] += ex2_approx(t0.y);
      a[(i + 2) & 7] += ex2_approx(t1.x);
      a[(i + 3) & 7] += ex2_approx(t1.y);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int r = r0 + i;
      if (r < p.R && k <= row_pos(p, r, n))
        a[i & 7] += ex2_approx(fmaf(__uint_as_float(rr[i]), c, lds1(nl + i)));
    }
  }
}

// ---- TMEM slot hand-off --------------------------------------------------
// A warpgroup waits for slot g to be filled, copies its part of the slot into
// registers, and releases the slot before doing any arithmetic, so the MMA of
// later tiles overlaps the exponentials.

__device__ __forceinline__ bool slot_acquire(const ScoreParams& p, const Smem& sm, uint32_t g,
                                             bool ok) {
  if (ok && !wait_bar(&sm.tfull[g % kSlots], (g / kSlots) & 1, p)) ok = false;
  ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld needs the whole warp
  if (ok) tc_fence_after();
  return ok;
}

__device__ __forceinline__ void slot_release(const Smem& sm, uint32_t g) {
  tc_fence_before();
  mbar_arrive(&sm.tempty[g % kSlots]);
}

template <int NCH>
__device__ __forceinline__ void load_slot(uint32_t taddr, uint32_t (&r)[NCH][32]) {
#pragma unroll
  for (int c = 0; c < NCH; ++c) tmem_ld32_async(taddr + c * 32, r[c]);
#pragma unroll
  for (int c = 0; c < NCH; ++c) tmem_wait32(r[c]);
}

// Sweep 1, slot g: this thread's row `row` against the tile's 128 keys, in two
// 64-column pieces (copy, then arithmetic); the slot is released after the
// second copy.
__device__ __forceinline__ void s1_slot(const ScoreParams& p, const Smem& sm, uint32_t lane_addr,
                                        uint32_t g, bool& ok, int row, int n, int kb, float& m,
                                        float& z) {
  ok = slot_acquire(p, sm, g, ok);
  const int tr = row < p.R ? row_pos(p, row, n) : -1;
  const bool full = (kb + kTileKeys - 1) <= (n - p.W);  // every key visible to every row
#pragma unroll
  for (int piece = 0; piece < 2; ++piece) {
    // Loaded even when the wait failed (the address is always inside this
    // CTA's TMEM allocation; the values are then discarded): a conditional
    // load would leave the array undefined on one path and spill it.
    uint32_t r[2][32];
    load_slot<2>(lane_addr + piece * 64, r);
    if (piece == 1) slot_release(sm, g);
    if (ok && tr >= 0) {
      s1_chunk(r[0], p.scale_log2, full, kb + piece * 64, tr, m, z);
      s1_chunk(r[1], p.scale_log2, full, kb + piece * 64 + 32, tr, m, z);
    }
  }
}

// Sweep 2, slot g: this thread's key k against rows r0 .. r0 + 32*nch, in
// pieces of up to 64 columns; partial sum into a[8].
template <int NCH>
__device__ __forceinline__ void s2_piece(const ScoreParams& p, uint32_t taddr, bool ok, bool full,
                                         const float* nl, int r0, int k, int n, float (&a)[8]) {
  uint32_t r[NCH][32];
  load_slot<NCH>(taddr, r);
  if (!ok || k >= n) return;
#pragma unroll
  for (int c = 0; c < NCH; ++c) s2_chunk(p, r[c], full, nl + c * 32, r0 + c * 32, k, n, a);
}

__device__ __forceinline__ void s2_slot(const ScoreParams& p, const Smem& sm, uint32_t lane_addr,
                                        uint32_t g, bool& ok, int nch, int r0, int k, int n,
                                        int kb, const float* nlam, float (&a)[8]) {
  ok = slot_acquire(p, sm, g, ok);
  const bool full = (kb + kTileKeys - 1 <= n - p.W) && (r0 + nch * 32 <= p.R);
  for (int c = 0; c < nch; c += 2) {
    if (c + 1 < nch)
      s2_piece<2>(p, lane_addr + c * 32, ok, full, nlam + r0 + c * 32, r0 + c * 32, k, n, a);
    else
      s2_piece<1>(p, lane_addr + c * 32, ok, full, nlam + r0 + c * 32, r0 + c * 32, k, n, a);
  }
  slot_release(sm, g);
}

// Softmax warpgroup wg (0..3) owns TMEM slot wg.  Slot g of the tile stream
// (tile t, 128-row group h -> g = t*nh + h) lands in slot g % 4, so with
// nh = 2 warpgroup wg handles row group wg & 1 of the tiles t = wg >> 1 (mod 2)
// and with nh = 1 the whole of tiles t = wg (mod 4).  No two warpgroups
// share a slot or synchronise with each other; partial results go to global
// memory (sweep 1: per-row (max, sum) per warpgroup; sweep 2: one partial sum
// per 128-row group, added by the selection kernel).
__device__ __forceinline__ void softmax_wg(const ScoreParams& p, const Smem& sm, uint32_t tmem_base,
                                           int wg, int first, int stride, int J) {
  const int warp = threadIdx.x >> 5;
  const int quarter = warp & 3;                       // TMEM lane quarter of this warp
  const int lrow = quarter * 32 + (threadIdx.x & 31);  // TMEM lane: row (sweep 1) / key (sweep 2)
  const int wtid = threadIdx.x - (4 + 4 * wg) * 32;    // 0..127 within the warpgroup
  const int bar_id = 1 + wg;
  const int nh = p.R_pad > 128 ? 2 : 1;                // 128-row groups (slots) per tile
  const int half = nh == 2 ? (wg & 1) : 0;             // row group of this warpgroup
  const uint32_t tmask = nh == 2 ? 1 : 3, tres = nh == 2 ? (wg >> 1) : wg;  // own tiles: (t & tmask) == tres
  const int row = half * 128 + lrow;                   // sweep-1 row of this thread
  const int r0 = half * 128;                           // sweep-2 first row
  const int nch = (nh == 2 ? (half == 0 ? 128 : p.R_pad - 128) : p.R_pad) / 32;
  const int PR = nh == 2 ? 128 : p.R_pad;              // rows per sweep-1 partial record
  float* raw_out = half == 0 ? p.raw : p.raw1;
  const uint32_t lane_addr =
      tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + wg * kSlotCols;
  float* nlam = sm.lam + wg * p.R_pad;  // -lse2 of the current sweep-2 unit
  uint32_t tile = 0;
  bool ok = true;

  for (int j = 0; j <= J; ++j) {
    prefetch_item(p, first, stride, j, J);
    // ---------------- sweep 1 of item j ----------------
    if (j < J) {
      const int t = first + j * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      float m = -INFINITY, z = 0.f;
      for (int i = 0; i < it.ntiles; ++i) {
        const uint32_t gt = tile + i;
        if ((gt & tmask) != tres) continue;
        s1_slot(p, sm, lane_addr, gt * nh + half, ok, row, it.n, it.key0 + i * kTileKeys, m, z);
      }
      tile += it.ntiles;
      // publish this warpgroup's (max, sum) partial of the chunk: entry
      // [t][wg][lrow] of rows PR = 128 (two row groups) or R_pad (one)
      if (row < p.R_pad)
        p.part[(static_cast<size_t>(t) * kSoftmaxWGs + wg) * PR + lrow] = make_float2(m, z);
      __threadfence();
      named_bar_sync(bar_id, 128);
      if (wtid == 0) {
        const int old = atomicAdd(&p.cnt[it.u], 1);
        __threadfence();
        sm.flag[wg] = (old == kSoftmaxWGs * it.nchunks - 1);
      }
      named_bar_sync(bar_id, 128);
      if (sm.flag[wg]) {
        // Last arrival for this unit: merge every chunk's partials of each row
        // into lse2 = M + log2(Z), one pass, eight independent loads in flight.
        for (int r = wtid; r < p.R_pad; r += 128) {
          // entries of row r: one per warpgroup and chunk, of which only the
          // two warpgroups of r's row group wrote when nh = 2
          const int per_chunk = nh == 2 ? 2 : kSoftmaxWGs;
          const int nq = per_chunk * it.nchunks;
          const float2* base =
              p.part + static_cast<size_t>(it.cs) * kSoftmaxWGs * PR + (nh == 2 ? (r & 127) : r);
          float M = -INFINITY, Z = 0.f;
          for (int q0 = 0; q0 < nq; q0 += 8) {
            float2 e[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int q = q0 + i;
              // chunk q / per_chunk, warpgroup: nh=2 -> (r >> 7) + 2*(q & 1); nh=1 -> q & 3
              const int w = nh == 2 ? ((r >> 7) + 2 * (q & 1)) : (q & 3);
              e[i] = q < nq ? __ldcg(&base[(static_cast<size_t>(q / per_chunk) * kSoftmaxWGs + w) * PR])
                            : make_float2(-INFINITY, 0.f);
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              if (e[i].x == -INFINITY) continue;
              if (e[i].x > M) {
                Z = Z * ex2_approx(M - e[i].x) + e[i].y;
                M = e[i].x;
              } else {
                Z += e[i].y * ex2_approx(e[i].x - M);
              }
            }
          }
          p.lam[static_cast<size_t>(it.u) * p.R_pad + r] =
              (M == -INFINITY || Z <= 0.f) ? INFINITY : M + lg2_approx(Z);
        }
        __threadfence();
        named_bar_sync(bar_id, 128);
        if (wtid == 0 && it.u != p.stall_unit) st_release(&p.ready[it.u], 1);
      }
    }
    // ---------------- sweep 2 of item j-1 ----------------
    if (j > 0) {
      const int t = first + (j - 1) * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      if (wtid == 0) {
        int ready = ld_acquire(&p.ready[it.u]);
        if (!ready) {
          const uint64_t t0 = globaltimer_ns();
          uint32_t spins = 0;
          while (!(ready = ld_acquire(&p.ready[it.u]))) {
            __nanosleep(64);
            if ((++spins & 15u) == 0) {
              if (ld_volatile(p.abort_flag)) break;
              if (globaltimer_ns() - t0 > static_cast<uint64_t>(p.wait_ns)) {
                atomicExch(p.abort_flag, 1);
                atomicOr(p.status, kStatusTimeout);
                break;
              }
            }
          }
        }
        sm.flag[4 + wg] = ready;
      }
      named_bar_sync(bar_id, 128);
      const bool have = sm.flag[4 + wg] != 0;
      for (int r = r0 + wtid; r < r0 + nch * 32; r += 128)  // stored negated: exp2(s*c + (-lse2))
        nlam[r] = have ? -__ldcg(&p.lam[static_cast<size_t>(it.u) * p.R_pad + r]) : -INFINITY;
      named_bar_sync(bar_id, 128);
      float* out = raw_out + static_cast<size_t>(it.u) * p.S_cap;
      for (int i = 0; i < it.ntiles; ++i) {
        const uint32_t gt = tile + i;
        if ((gt & tmask) != tres) continue;
        const int kb = it.key0 + i * kTileKeys;
        const int k = kb + lrow;
        float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        s2_slot(p, sm, lane_addr, gt * nh + half, ok, nch, r0, k, it.n, kb, nlam, a);
        if (ok && k < it.n) out[k] = sum8(a) * p.inv_G;
      }
      tile += it.ntiles;
    }
  }
}

template <int D>
__global__ void __launch_bounds__(kScoreThreads, 1) score_kernel(const __grid_constant__ ScoreParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {  // the 128-byte swizzle needs 1024-byte aligned tiles
    if (threadIdx.x == 0) atomicOr(p.status, kStatusDevice);
    return;
  }
  const Smem sm = carve(smem_raw, p, D);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < p.stages; ++i) {
      mbar_init(&sm.kfull[i], 1);
      mbar_init(&sm.kempty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.qfull[i], 1);
      mbar_init(&sm.qempty[i], 1);
    }
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&sm.tfull[i], 1);
      mbar_init(&sm.tempty[i], 128);  // the 128 threads of the warpgroup that owns the tile
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

  const int total = p.chunk_start[p.n_units];
  const int first = blockIdx.x, stride = gridDim.x;
  const int J = first < total ? (total - first + stride - 1) / stride : 0;

  if (warp < 4) {
    regs_dealloc<kRegsControl>();
    if (warp == 0 && (threadIdx.x & 31) == 0) producer<D>(p, sm, first, stride, J);
    if (warp == 1) mma_issuer<D>(p, sm, tmem_base, first, stride, J);  // whole warp
  } else {
    regs_alloc<kRegsSoftmax>();
    softmax_wg(p, sm, tmem_base, (warp - 4) >> 2, first, stride, J);  // warpgroups 0..3
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kSlots * kSlotCols);
  }
}

// ---------------------------------------------------------------------------
// Prologue: per-unit chunk counts, prefix sums, item -> unit map, flag reset.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) prologue_kernel(const __grid_constant__ PrologueParams p) {
  __shared__ int warp_sums[32];
  __shared__ int carry;
  const int tid = threadIdx.x;
  if (tid == 0) {
    carry = 0;
    *p.abort_flag = 0;
  }
  for (int s = tid; s < p.B; s += blockDim.x) {
    int n = p.lens_in[s];
    if (n < 0 || n > p.S_cap) {
      atomicOr(p.status, kStatusDevice);
      n = 0;
    }
    p.lens[s] = n;
  }
  __syncthreads();
  const int per_layer = p.B * p.H_kv;
  for (int base = 0; base < p.n_units; base += blockDim.x) {
    const int u = base + tid;
    int c = 0;
    if (u < p.n_units) {
      const int ls = u / per_layer;
      const int s = (u - ls * per_layer) / p.H_kv;
      const int n = p.lens[s];
      const bool need = n > 0 && (p.slayer_method[ls] == KVEV_H2O || n > p.slayer_budget[ls]);
      c = need ? (n + p.chunk_keys - 1) / p.chunk_keys : 0;
      p.cnt[u] = 0;
      p.ready[u] = 0;
    }
    // block-wide exclusive scan of c
    int x = c;
    const int lane = tid & 31, w = tid >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[w] = x;
    __syncthreads();
    if (w == 0) {
      int ws = lane < (int)(blockDim.x >> 5) ? warp_sums[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, ws, o);
        if (lane >= o) ws += y;
      }
      warp_sums[lane] = ws;
    }
    __syncthreads();
    const int excl = carry + (w > 0 ? warp_sums[w - 1] : 0) + x - c;
    if (u < p.n_units) {
      p.chunk_start[u] = excl;
      const int n = p.lens[(u % per_layer) / p.H_kv];
      for (int q = 0; q < c; ++q) {
        const int key0 = q * p.chunk_keys;
        const int nk = min(p.chunk_keys, n - key0);
        const int ntiles = (nk + kTileKeys - 1) / kTileKeys;
        p.item[excl + q] = make_int4(u, n, key0, ntiles | (c << 16));
      }
    }
    __syncthreads();
    if (tid == blockDim.x - 1) carry = excl + c;
    __syncthreads();
  }
  if (tid == 0) p.chunk_start[p.n_units] = carry;
}

}  // namespace

int score_smem_bytes(int d, int q_rows, int R_pad, int stages) {
  size_t off = 0;
  off += 2 * static_cast<size_t>(q_rows) * d * 2;
  off += static_cast<size_t>(stages) * kTileKeys * d * 2;
  off += kSoftmaxWGs * sizeof(float) * R_pad;
  off = (off + 7) & ~size_t(7);
  off += sizeof(uint64_t) * (2 * stages + 4 + 2 * kSlots + 1);
  off += sizeof(uint32_t) + 8 * sizeof(int);
  return static_cast<int>((off + 127) & ~size_t(127));
}

int score_kernel_regs(int d) {
  cudaFuncAttributes a = {};
  const cudaError_t e = d == 64 ? cudaFuncGetAttributes(&a, score_kernel<64>)
                                : cudaFuncGetAttributes(&a, score_kernel<128>);
  return e == cudaSuccess ? a.numRegs : -1;
}

cudaError_t score_set_smem(int d, size_t smem) {
  if (d == 64)
    return cudaFuncSetAttribute(score_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem));
  return cudaFuncSetAttribute(score_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(smem));
}

cudaError_t launch_prologue(const PrologueParams& p, cudaStream_t s) {
  prologue_kernel<<<1, 1024, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_score(const ScoreParams& p, int d, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kScoreThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // all CTAs co-resident
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (d == 64) return cudaLaunchKernelEx(&cfg, score_kernel<64>, p);
  return cudaLaunchKernelEx(&cfg, score_kernel<128>, p);
}

}  // namespace kvev
