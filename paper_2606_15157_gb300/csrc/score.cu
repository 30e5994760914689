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
// Work items are chunks of chunk_keys keys (an even number of 128-key tiles,
// swept in 256-key super-tiles).  A CTA runs sweep 1 of item j + kLag before
// sweep 2 of item j, so the unit's normaliser, which needs every chunk of the
// unit (some on other CTAs), is almost always published by the time sweep 2
// needs it.  The chunk whose partials complete the unit's merge tree publishes
// lse2 (release flag); sweep-2 readers wait on it with a time bound.  All CTAs
// are co-resident (cooperative launch) and a unit spans at most two rounds of
// items, so the wait always ends.
//
// Roles per CTA (640 threads, five warpgroups): warp 0 issues TMA loads (one
// thread); warp 1 owns TMEM and issues tcgen05.mma (an elected lane); warp 2
// publishes each chunk's row partials and climbs the unit's merge tree; warp 3
// stages -lse2 for sweep 2; warpgroups 1-4 are softmax warpgroups.  The tensor
// core fills 256-column TMEM units (two adjacent 128-column slots) in a ring
// of two: sweep 1 one unit per (super-tile, 128-row group), sweep 2 one unit
// per 128-key tile.  All four softmax warpgroups consume every unit, 64
// columns each, copying them with one tcgen05.ld and releasing the unit
// before any arithmetic.  setmaxnreg moves registers from warpgroup 0 to the
// softmax warpgroups.
#include "score_common.cuh"

namespace kvev {

namespace {

struct Smem {
  uint8_t* qbuf;     // q_bufs Q buffers of qbytes each, indexed arithmetically (a dynamically
  uint32_t qbytes;   // indexed member array would push the whole struct to local memory)
  uint8_t* kbuf;     // stages * tile bytes
  float* lam;        // [2][R_pad]: -lse2 of the units of the next two sweep-2 entries
  float* red;        // [kSoftmaxWGs][kRedTiles][128]: per-warpgroup partial key sums of a batch
                     // of sweep-2 tiles
  float2* pc;        // [kSoftmaxWGs][R_pad]: per-warpgroup (max, sum) of a sweep-1 item
  uint64_t* lfull;   // [2] lam buffer written by the normaliser warp
  uint64_t* lempty;  // [2] lam buffer read by the softmax warpgroups
  uint64_t* pfull;   // partials of a sweep-1 entry written to pc by the softmax threads
  uint64_t* pempty;  // pc read by the publisher warp
  uint64_t* kfull;
  uint64_t* kempty;
  uint64_t* qfull;
  uint64_t* qempty;
  uint64_t* tfull;
  uint64_t* tempty;
  uint64_t* done;
  uint32_t* tmem_slot;
  uint64_t* nap;     // never completed: the normaliser warp sleeps on it between polls
};

__host__ __device__ __forceinline__ size_t smem_size(int D, int q_rows, int q_bufs, int R_pad, int stages,
                                                      size_t* koff, size_t* loff, size_t* roff,
                                                      size_t* poff, size_t* boff) {
  size_t off = static_cast<size_t>(q_bufs) * q_rows * D * 2;
  *koff = off;
  off += static_cast<size_t>(stages) * kSuperKeys * D * 2;
  *loff = off;
  off += sizeof(float) * 2 * R_pad;
  *roff = off;
  off += sizeof(float) * kSoftmaxWGs * kRedTiles * 128;
  off = (off + 7) & ~size_t(7);
  *poff = off;
  off += sizeof(float2) * kSoftmaxWGs * R_pad;
  *boff = off;
  off += sizeof(uint64_t) * (2 * stages + 4 + 2 * kSlots + 1 + 7);
  off += sizeof(uint32_t);
  return off;
}

__device__ __forceinline__ Smem carve(uint8_t* base, const ScoreParams& p, int D) {
  Smem s;
  size_t koff, loff, roff, poff, boff;
  smem_size(D, p.q_rows, p.q_bufs, p.R_pad, p.stages, &koff, &loff, &roff, &poff, &boff);
  s.qbuf = base;
  s.qbytes = static_cast<uint32_t>(p.q_rows) * D * 2;
  s.kbuf = base + koff;
  s.lam = reinterpret_cast<float*>(base + loff);
  s.red = reinterpret_cast<float*>(base + roff);
  s.pc = reinterpret_cast<float2*>(base + poff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + boff);
  s.kfull = bars;
  s.kempty = bars + p.stages;
  s.qfull = bars + 2 * p.stages;
  s.qempty = s.qfull + 2;
  s.tfull = s.qempty + 2;
  s.tempty = s.tfull + kSlots;
  s.done = s.tempty + kSlots;
  s.lfull = s.done + 1;
  s.lempty = s.lfull + 2;
  s.pfull = s.lempty + 2;
  s.pempty = s.pfull + 1;
  s.nap = s.pempty + 1;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.nap + 1);
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

// A CTA's work entries in order: at step j = 0 .. J + kLag - 1, sweep 1 of
// item j (j < J), then sweep 2 of item j - kLag (j >= kLag).  Sweep 2 of an
// item runs kLag sweep-1 items after its own sweep 1, so the unit's row
// normalisers (which need every chunk of the unit, some of them on other
// CTAs) are almost always published by then.  With the normalisers supplied
// (single sweep), the entries are sweep 2 of items 0 .. J-1.  Every entry
// loads its own Q (buffer e mod 2 for entry e).
constexpr int kLag = 2;
struct EntryIter {
  int J, j = 0, sweep = -1;
  bool single;
  __device__ __forceinline__ EntryIter(int J_, bool single_) : J(J_), single(single_) {}
  // Next entry: item index jj (of this CTA) and sweep; false at the end.
  __device__ __forceinline__ bool next(int& jj, int& sw) {
    if (single) {
      if (++sweep >= J) return false;
      jj = sweep;
      sw = 1;
      return true;
    }
    for (;;) {
      if (++sweep == 2) {
        sweep = 0;
        ++j;
      }
      if (j >= J + kLag) return false;
      jj = sweep == 0 ? j : j - kLag;
      if (jj >= 0 && jj < J) {
        sw = sweep;
        return true;
      }
    }
  }
};

// ---------------------------------------------------------------------------
// Producer: TMA loads of Q (once per item) and of K tiles (twice per item).
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void load_q(const ScoreParams& p, const Smem& sm, uint32_t e, const ItemInfo& it) {
  const uint32_t qb = e % p.q_bufs;
  mbar_expect_tx(&sm.qfull[qb], static_cast<uint32_t>(p.R_pad) * D * 2);
  const int qrow = (it.s * p.H_q + it.h * p.G) * p.W;
#pragma unroll
  for (int kc = 0; kc < D / 64; ++kc)
    tma_load_2d(sm.qbuf + qb * sm.qbytes + static_cast<size_t>(kc) * p.q_rows * 128, &p.qmap[it.ls],
                kc * 64, qrow, &sm.qfull[qb]);
}

template <int D>
__device__ __forceinline__ void producer(const ScoreParams& p, const Smem& sm, int first, int stride, int J) {
  constexpr uint32_t kStageBytes = kSuperKeys * D * 2;
  const uint64_t keep = policy_evict_last();   // first read of a K tile: keep it for the re-read
  const uint64_t drop = policy_evict_first();  // second read: its last use
  uint32_t tile = 0;            // super-tiles issued (for the drain after an abort)
  uint32_t pst = 0, pph = 0;    // K stage ring: position and phase of the next tile
  uint32_t q_issued = 0;        // entries whose Q load has been issued
  const uint32_t nq = p.q_bufs;
  // Q of entry x goes into buffer x mod nq once entry x - nq has released it
  auto q_free = [&](uint32_t x) { return mbar_try_wait(&sm.qempty[x % nq], ((x / nq) & 1) ^ 1); };
  bool ok = true;
  EntryIter ei(J, p.single != 0);
  int jj, sw;
  for (uint32_t e = 0; ok && ei.next(jj, sw); ++e) {
    const int t = first + jj * stride;
    if (sw == 0) prefetch_item(p, first, stride, jj, J);
    const ItemInfo it = decode_item(p, t, load_item(p, t));
    EntryIter la = ei;
    int jn, swn;
    const bool has_next = la.next(jn, swn);
    const CUtensorMap* kmap = &p.kmap[it.ls];
    const int row0 = (it.s * p.H_kv + it.h) * p.S_cap + it.key0;
    const int nst = (it.ntiles + 1) / 2;  // 256-key super-tiles of the item
    // This entry's Q goes out as soon as its buffer is free, and at the
    // latest before the super-tile that fills the last stage (the K loads
    // before it do not depend on Q, so they stream in meanwhile); with two
    // buffers the next entry's Q goes out during this entry.
    const int q_by = min(p.stages, nst) - 1;
    for (int i = 0; i < nst; ++i, ++tile) {
      if (q_issued == e && (i >= q_by || q_free(e))) {
        if (!wait_bar(&sm.qempty[e % nq], ((e / nq) & 1) ^ 1, p)) { ok = false; break; }
        load_q<D>(p, sm, e, it);
        ++q_issued;
      }
      if (nq > 1 && has_next && q_issued == e + 1 && q_free(e + 1)) {
        const int tn = first + jn * stride;
        load_q<D>(p, sm, e + 1, decode_item(p, tn, load_item(p, tn)));
        ++q_issued;
      }
      const uint32_t st = pst, ph = pph;
      if (++pst == static_cast<uint32_t>(p.stages)) { pst = 0; pph ^= 1; }
      if (!wait_bar(&sm.kempty[st], ph ^ 1, p)) { ok = false; break; }
      uint8_t* dst = sm.kbuf + static_cast<size_t>(st) * kStageBytes;
      mbar_expect_tx(&sm.kfull[st], kStageBytes);
#pragma unroll
      for (int kc = 0; kc < D / 64; ++kc)
        tma_load_2d_hint(dst + kc * (kSuperKeys * 128), kmap, kc * 64, row0 + i * kSuperKeys,
                         &sm.kfull[st], sw == 0 ? keep : drop);
    }
  }
  // Drain: make sure no copy is still landing in shared memory when the CTA
  // retires (only relevant after an abort; normally every load was consumed).
  if (!ok) {
    const uint32_t S = p.stages;
    for (uint32_t st = 0; st < S && st < tile; ++st) {
      const uint32_t last = ((tile - 1 - st) / S) * S + st;  // last tile issued into st
      wait_bar_drain(&sm.kfull[st], (last / S) & 1, 100000000ull);
    }
    for (uint32_t b = 0; b < nq && b < q_issued; ++b) {
      const uint32_t last = ((q_issued - 1 - b) / nq) * nq + b;  // last Q load into buffer b
      wait_bar_drain(&sm.qfull[b], (last / nq) & 1, 100000000ull);
    }
  }
}

// ---------------------------------------------------------------------------
// MMA issuer (one warp; an elected lane issues): sweep 1 -> S = Q K^T,
// sweep 2 -> S^T = K Q^T.
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void mma_issuer(const ScoreParams& p, const Smem& sm, uint32_t tmem_base, int first,
                           int stride, int J) {
  constexpr uint32_t kStageBytes = kSuperKeys * D * 2;
  const int nh = p.R_pad > 128 ? 2 : 1;
  // sweep 1: S[128 rows of a group][256 keys of a super-tile]
  const uint32_t idesc1 = idesc_bf16_f32(128, kSuperKeys);
  // sweep 2: S^T[128 keys][every window row] (up to 256)
  const uint32_t idesc2 = idesc_bf16_f32(128, p.R_pad);
  // descriptor steps (address / 16) between the 64-wide column blocks of Q and of a K stage
  const uint32_t qcol_step = static_cast<uint32_t>(p.q_rows) * 128 / 16;
  constexpr uint32_t kcol_step = kSuperKeys * 128 / 16;
  constexpr uint32_t khalf = kTileKeys * 128 / 16;   // second 128-key half of a super-tile
  constexpr uint32_t qgroup = 128 * 128 / 16;         // second 128-row group of Q
  uint32_t st = 0, kph = 0;  // K stage ring: position and phase of the next super-tile
  uint32_t sl = 0, tph = 0;  // TMEM ring of two 256-column units: first slot and phase
  bool ok = true;
  EntryIter ei(J, p.single != 0);
  int jj, sw;
  for (uint32_t e = 0; ok && ei.next(jj, sw); ++e) {
    const int t = first + jj * stride;
    if (sw == 0) prefetch_item(p, first, stride, jj, J);
    const ItemInfo it = decode_item(p, t, load_item(p, t));
    const uint32_t qb = e % p.q_bufs;
    const uint64_t qdesc0 = sw128_desc(smem_u32(sm.qbuf) + qb * sm.qbytes);
    if (!wait_bar_warp(&sm.qfull[qb], (e / p.q_bufs) & 1, p)) { ok = false; break; }
    const bool s1 = sw == 0;
    const int nst = (it.ntiles + 1) / 2;
    for (int j = 0; ok && j < nst; ++j) {
      if (!wait_bar_warp(&sm.kfull[st], kph, p)) { ok = false; break; }
      // Descriptors built once per super-tile: a descriptor's low field is
      // the address / 16, so the k-step offsets (all inside shared memory, no
      // carry out of the field) are plain adds.
      const uint64_t kdesc = sw128_desc(smem_u32(sm.kbuf) + st * kStageBytes);
      // Work units of one super-tile, each a 256-column TMEM unit (two
      // slots) with one full and one empty barrier (those of its first
      // slot): sweep 1 -> one unit per 128-row group of Q, N = 256 keys;
      // sweep 2 -> one unit per 128-key half, N = every window row.
      const int nu = s1 ? nh : min(2, it.ntiles - 2 * j);
      for (int u = 0; u < nu; ++u) {
        if (!wait_bar_warp(&sm.tempty[sl], tph ^ 1, p)) { ok = false; break; }
        tc_fence_after();
        const uint32_t dcol = tmem_base + sl * kSlotCols;
        if (s1) {
          const uint64_t qdesc = qdesc0 + static_cast<uint64_t>(u * qgroup);
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint32_t a = (k >> 2) * qcol_step + (k & 3) * 2, b = (k >> 2) * kcol_step + (k & 3) * 2;
            umma_bf16_elect(dcol, qdesc + a, kdesc + b, idesc1, k > 0);
          }
        } else {
          const uint64_t adesc = kdesc + static_cast<uint64_t>(u * khalf);
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint32_t a = (k >> 2) * kcol_step + (k & 3) * 2, b = (k >> 2) * qcol_step + (k & 3) * 2;
            umma_bf16_elect(dcol, adesc + a, qdesc0 + b, idesc2, k > 0);
          }
        }
        umma_commit_elect(&sm.tfull[sl]);
        sl += 2;
        if (sl == kSlots) { sl = 0; tph ^= 1; }
      }
      if (!ok) break;
      umma_commit_elect(&sm.kempty[st]);
      if (++st == static_cast<uint32_t>(p.stages)) { st = 0; kph ^= 1; }
    }
    if (ok) umma_commit_elect(&sm.qempty[qb]);  // the entry's Q buffer is free once these finish
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


__device__ __forceinline__ void s2_chunk(const ScoreParams& p, const uint32_t (&rr)[32], bool full,
                                         const float* nl, int r0, int k, int n, float2 (&a)[4]) {
  const float c = p.scale_log2;
  if (full) {
    s2_chunk_full(rr, c, nl, a);
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const int r = r0 + i;
      if (r < p.R && k <= row_pos(p, r, n)) {
        const float e = ex2_approx(fmaf(__uint_as_float(rr[i]), c, lds1(nl + i)));
        if (i & 1) a[(i >> 1) & 3].y += e; else a[(i >> 1) & 3].x += e;
      }
    }
  }
}

// ---- TMEM unit hand-off ----------------------------------------------------
// Every 256-column unit is consumed by all four softmax warpgroups:
// warpgroup w copies its 64 columns and releases the unit at once (the
// unit's empty barrier counts the 16 softmax warps: one elected lane arrives
// for its warp, as a shared-memory barrier takes its arrivals one at a time),
// so the tensor core refills it as soon as the last slice is copied and no
// warpgroup holds TMEM while it computes.

__device__ __forceinline__ bool slot_wait(const ScoreParams& p, const Smem& sm, uint32_t g, bool ok) {
  if (ok && !wait_bar(&sm.tfull[g & (kSlots - 1)], (g / kSlots) & 1, p)) ok = false;
  return ok;
}


// This warpgroup's 64 columns of a unit (the unit's two slots are 256
// adjacent columns; warpgroup w takes [64w, 64w + 64)) in one load, released
// (through the first slot's barrier) before any arithmetic.
__device__ __forceinline__ void unit_take(const Smem& sm, uint32_t lane_base, uint32_t g, uint32_t (&r0)[32],
                                          uint32_t (&r1)[32]) {
  const uint32_t s0 = g & (kSlots - 1);
  tmem_ld64_async(lane_base + s0 * kSlotCols, r0, r1);
  tmem_wait64(r0, r1);
  tc_fence_before();
  __syncwarp();
  mbar_arrive_elect(&sm.tempty[s0]);
}

__device__ __forceinline__ void softmax_wg(const ScoreParams& p, const Smem& sm, uint32_t tmem_base,
                                           int wg, int first, int stride, int J) {
  const int warp = threadIdx.x >> 5;
  const int quarter = warp & 3;                        // TMEM lane quarter of this warp
  const int lrow = quarter * 32 + (threadIdx.x & 31);  // TMEM lane: row (sweep 1) / key (sweep 2)
  const int stid = threadIdx.x - 128;                  // 0..511 over the softmax warpgroups
  const int nh = p.R_pad > 128 ? 2 : 1;                // 128-row groups (slots) per tile
  // this warpgroup's 64 columns of every 256-column unit
  const uint32_t lane_base =
      tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(64 * wg);
  // sweep 2: this warpgroup's rows [64wg, 64wg + 32) and [64wg + 32, 64wg + 64)
  const int r0a = 64 * wg, r0b = 64 * wg + 32;
  const bool has_a = r0a < p.R_pad;
  const bool has_b = r0b < p.R_pad;
  uint32_t g = 0;     // slot stream position (advances 2 per 256-column unit)
  uint32_t q1 = 0, q2 = 0;  // sweep-1 / sweep-2 entries done
  bool ok = true;

  EntryIter ei(J, p.single != 0);
  int jj, sw;
  while (ei.next(jj, sw)) {
    // ---------------- sweep 1 ----------------
    if (sw == 0) {
      prefetch_item(p, first, stride, jj, J);
      const int t = first + jj * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      float m0 = -INFINITY, z0 = 0.f, m1 = -INFINITY, z1 = 0.f;
      const int tr0 = lrow < p.R ? row_pos(p, lrow, it.n) : -1;
      const int tr1 = 128 + lrow < p.R ? row_pos(p, 128 + lrow, it.n) : -1;
      // One unit per (256-key super-tile, 128-row group): this warpgroup's 32
      // keys of each 128-key half, for the thread's row of the group.  Rows
      // that do not exist (tr < 0) are computed like the others and dropped
      // when the warpgroup publishes.
      const int nst = (it.ntiles + 1) / 2;
      for (int j = 0; j < nst; ++j) {
        const int kb = it.key0 + j * kSuperKeys;
        const int k0 = kb + 64 * wg;                       // keys k0 .. k0 + 63
        const bool full = kb + kSuperKeys - 1 <= it.n - p.W;  // every key visible to every row
        for (int h = 0; h < nh; ++h) {
          ok = slot_wait(p, sm, g, ok);
          uint32_t r0[32], r1[32];
          unit_take(sm, lane_base, g, r0, r1);
          float v0[32], v1[32];
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            v0[q] = __uint_as_float(r0[q]);
            v1[q] = __uint_as_float(r1[q]);
          }
          const int tr = h == 0 ? tr0 : tr1;
          if (!full) {
            mask_chunk(v0, k0, tr);
            mask_chunk(v1, k0 + 32, tr);
          }
          if (h == 0)
            s1_chunk64(v0, v1, p.scale_log2, m0, z0);
          else
            s1_chunk64(v0, v1, p.scale_log2, m1, z1);
          g += 2;
        }
      }
      // hand the four warpgroups' (max, sum) of each row to the publisher warp
      if (!wait_bar(&sm.pempty[0], (q1 & 1) ^ 1, p)) ok = false;
      const float2 none = make_float2(-INFINITY, 0.f);
      if (lrow < p.R_pad) sm.pc[wg * p.R_pad + lrow] = tr0 >= 0 && ok ? make_float2(m0, z0) : none;
      if (nh == 2 && 128 + lrow < p.R_pad)
        sm.pc[wg * p.R_pad + 128 + lrow] = tr1 >= 0 && ok ? make_float2(m1, z1) : none;
      __syncwarp();
      mbar_arrive_elect(&sm.pfull[0]);
      ++q1;
    }
    // ---------------- sweep 2 ----------------
    else {
      const int t = first + jj * stride;
      const ItemInfo it = decode_item(p, t, load_item(p, t));
      // -lse2 of the unit, loaded ahead by the normaliser warp
      const uint32_t lb = q2 & 1;
      if (!wait_bar(&sm.lfull[lb], (q2 >> 1) & 1, p)) ok = false;
      const float* lam = sm.lam + lb * p.R_pad;
      float* out = p.raw + static_cast<size_t>(it.u) * p.S_cap;
      for (int i = 0; i < it.ntiles; ++i) {
        const int kb = it.key0 + i * kTileKeys;
        const int k = kb + lrow;
        const bool key_full = kb + kTileKeys - 1 <= it.n - p.W;
        float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                       make_float2(0.f, 0.f)};
        ok = slot_wait(p, sm, g, ok);
        {
          uint32_t ra[32], rb[32];
          unit_take(sm, lane_base, g, ra, rb);
          if (ok && key_full && r0b + 32 <= p.R) {  // the common case: every key and row counts
            s2_chunk_full(ra, p.scale_log2, lam + r0a, a);
            s2_chunk_full(rb, p.scale_log2, lam + r0b, a);
          } else {
            if (ok && has_a && k < it.n)
              s2_chunk(p, ra, key_full && r0a + 32 <= p.R, lam + r0a, r0a, k, it.n, a);
            if (ok && has_b && k < it.n)
              s2_chunk(p, rb, key_full && r0b + 32 <= p.R, lam + r0b, r0b, k, it.n, a);
          }
        }
        g += 2;
        // Each warpgroup keeps its partial sum of every key of a batch of
        // kRedTiles tiles in its own shared-memory rows; at the end of the
        // batch all four are added (in warpgroup order) and stored, with one
        // barrier on either side instead of a hand-off per tile.
        const int bt = i % kRedTiles;
        sm.red[(wg * kRedTiles + bt) * 128 + lrow] = sum4x2(a);
        if (bt == kRedTiles - 1 || i == it.ntiles - 1) {
          named_bar_sync(1, 128 * kSoftmaxWGs);
          const int key0 = it.key0 + (i - bt) * kTileKeys;
          for (int q = stid; q < (bt + 1) * 128; q += 128 * kSoftmaxWGs) {
            float sum = 0.f;
#pragma unroll
            for (int w = 0; w < kSoftmaxWGs; ++w) sum += sm.red[w * kRedTiles * 128 + q];
            if (ok && key0 + q < it.n) out[key0 + q] = sum * p.inv_G;
          }
          // the batch's rows may be overwritten, and after the entry's last
          // batch every warpgroup is done reading lam
          named_bar_sync(1, 128 * kSoftmaxWGs);
        }
      }
      if (stid == 0) mbar_arrive(&sm.lempty[lb]);
      ++q2;
    }
  }
}

// ---------------------------------------------------------------------------
// Publisher warp: for each sweep-1 entry, merge the four warpgroups' (max,
// sum) of every row into the chunk's record, then climb the unit's merge tree:
// a node's record lives in the slot of its first leaf chunk; the last of a
// node's (up to kTreeFanIn) children to arrive merges its siblings' records
// into its own and carries the result one level up.  Whoever completes the
// root turns it into the unit's lse2 and releases it.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void publisher(const ScoreParams& p, const Smem& sm, int first, int stride, int J) {
  constexpr int kRowsPerLane = 8;  // R_pad <= 256
  const int lane = threadIdx.x & 31;
  const int nr = p.R_pad >> 5;
  uint32_t q1 = 0;
  EntryIter ei(J, p.single != 0);
  int jj, sw;
  while (ei.next(jj, sw)) {
    if (sw != 0) continue;
    const int t = first + jj * stride;
    const ItemInfo it = decode_item(p, t, load_item(p, t));
    if (!wait_bar_warp(&sm.pfull[0], q1 & 1, p)) return;
    float2 acc[kRowsPerLane];  // rows lane + 32 i of the current tree node
#pragma unroll
    for (int i = 0; i < kRowsPerLane; ++i) {
      acc[i] = make_float2(-INFINITY, 0.f);
      if (i < nr) {
#pragma unroll
        for (int w = 0; w < kSoftmaxWGs; ++w) acc[i] = merge_ms(acc[i], sm.pc[w * p.R_pad + lane + 32 * i]);
      }
    }
    __syncwarp();
    mbar_arrive_elect(&sm.pempty[0]);  // pc may be overwritten
    ++q1;
    int c = t - it.cs;         // index of the current node within its level (a leaf: the chunk)
    int nodes = it.nchunks;    // nodes of the current level
    int span = 1;              // leaf chunks under a node of the current level
    int level = 0;
    bool root = nodes == 1;
    while (!root) {
      float2* rec = p.part + static_cast<size_t>(it.cs + c * span) * p.R_pad;
#pragma unroll
      for (int i = 0; i < kRowsPerLane; ++i)
        if (i < nr) rec[lane + 32 * i] = acc[i];
      __threadfence();
      __syncwarp();
      const int c0 = c / kTreeFanIn * kTreeFanIn;  // first sibling
      const int nchild = min(kTreeFanIn, nodes - c0);
      int last = 0;
      if (lane == 0) {
        int* cnt = p.node_cnt + static_cast<size_t>(it.cs + c0 * span) * kTreeLevels + level;
        last = atomicAdd(cnt, 1) == nchild - 1;
        __threadfence();
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (!last) break;
      for (int k = 0; k < nchild; ++k) {
        if (c0 + k == c) continue;
        const float2* sib = p.part + static_cast<size_t>(it.cs + (c0 + k) * span) * p.R_pad;
#pragma unroll
        for (int h = 0; h < kRowsPerLane; h += 4) {  // four loads in flight (64 registers)
          float2 e[4];
#pragma unroll
          for (int i = 0; i < 4; ++i)
            e[i] = h + i < nr ? __ldcg(&sib[lane + 32 * (h + i)]) : make_float2(-INFINITY, 0.f);
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[h + i] = merge_ms(acc[h + i], e[i]);
        }
      }
      c /= kTreeFanIn;
      nodes = (nodes + kTreeFanIn - 1) / kTreeFanIn;
      span *= kTreeFanIn;
      ++level;
      root = nodes == 1;
    }
    if (!root) continue;
    // The root: lse2 = M + log2(Z) per row.
#pragma unroll
    for (int i = 0; i < kRowsPerLane; ++i) {
      if (i < nr)
        p.lam[static_cast<size_t>(it.u) * p.R_pad + lane + 32 * i] =
            (acc[i].x == -INFINITY || acc[i].y <= 0.f) ? INFINITY : acc[i].x + lg2_approx(acc[i].y);
    }
    __threadfence();
    __syncwarp();
    if (lane == 0 && it.u != p.stall_unit) st_release(&p.ready[it.u], 1);
  }
}

// ---------------------------------------------------------------------------
// Normaliser warp: for each sweep-2 entry, wait for the unit's lse2 (bounded)
// and copy -lse2 into the entry's lam buffer ahead of the softmax warpgroups.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void lam_loader(const ScoreParams& p, const Smem& sm, int first, int stride, int J) {
  const int lane = threadIdx.x & 31;
  uint32_t q2 = 0;
  EntryIter ei(J, p.single != 0);
  int jj, sw;
  while (ei.next(jj, sw)) {
    if (sw != 1) continue;
    const int t = first + jj * stride;
    const ItemInfo it = decode_item(p, t, load_item(p, t));
    const uint32_t lb = q2 & 1;
    if (!wait_bar_warp(&sm.lempty[lb], ((q2 >> 1) & 1) ^ 1, p)) return;
    // The whole warp polls the unit's flag; between polls it sleeps on a
    // shared-memory barrier that never completes (a suspended wait, which
    // unlike a spin leaves this warp's issue port to the softmax warps that
    // share it).  The normaliser is needed one entry later at the earliest,
    // so a microsecond between polls costs nothing.
    int ready = 0;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
      int v = 0, stop = 0;
      if (lane == 0) {
        v = ld_acquire(&p.ready[it.u]);
        if (!v && ld_volatile(p.abort_flag)) stop = 1;
        if (!v && !stop && globaltimer_ns() - t0 > static_cast<uint64_t>(p.wait_ns)) {
          atomicExch(p.abort_flag, 1);
          atomicOr(p.status, kStatusTimeout);
          stop = 1;
        }
      }
      ready = __shfl_sync(0xffffffffu, v, 0);
      if (ready || __shfl_sync(0xffffffffu, stop, 0)) break;
      mbar_try_wait_sleep(sm.nap, 0, 1000);
    }
    __syncwarp();  // the other lanes read lse2 after lane 0's acquire
    float* lam = sm.lam + lb * p.R_pad;
    for (int r = lane; r < p.R_pad; r += 32)  // stored negated: exp2(s*c + (-lse2))
      lam[r] = ready ? -__ldcg(&p.lam[static_cast<size_t>(it.u) * p.R_pad + r]) : -INFINITY;
    __syncwarp();
    mbar_arrive_elect(&sm.lfull[lb]);
    ++q2;
    if (!ready) return;
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
      mbar_init(&sm.tempty[i], 4 * kSoftmaxWGs);  // every softmax warp copies its slice
    }
    mbar_init(sm.done, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.lfull[i], 1);
      mbar_init(&sm.lempty[i], 1);
    }
    mbar_init(sm.pfull, 4 * kSoftmaxWGs);
    mbar_init(sm.pempty, 1);
    mbar_init(sm.nap, 1);
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
    if (warp == 2) publisher(p, sm, first, stride, J);                 // whole warp
    if (warp == 3) lam_loader(p, sm, first, stride, J);                // whole warp
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
// Each CTA takes a contiguous slice of the units: it scans the chunk counts
// of every unit up to the end of its slice (a few block-wide scans; the
// counts are cheap to recompute) and writes its units' start offsets, work
// items and cleared merge-tree counters, so that the writes are spread over
// the grid instead of queued behind one SM.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) prologue_kernel(const __grid_constant__ PrologueParams p) {
  __shared__ int warp_sums[32];
  __shared__ int carry;
  const int tid = threadIdx.x;
  const int slice = (p.n_units + gridDim.x - 1) / gridDim.x;
  const int u0 = min(static_cast<int>(blockIdx.x) * slice, p.n_units);
  const int u1 = min(u0 + slice, p.n_units);
  if (tid == 0) carry = 0;
  if (blockIdx.x == 0) {
    if (tid == 0) *p.abort_flag = 0;
    for (int s = tid; s < p.B; s += blockDim.x) {
      int n = p.lens_in[s];
      if (n < 0 || n > p.S_cap) {
        atomicOr(p.status, kStatusDevice);
        n = 0;
      }
      p.lens[s] = n;
    }
  }
  __syncthreads();
  if (u0 == u1) {  // an empty slice (or no scoring units at all)
    if (p.n_units == 0 && blockIdx.x == 0 && tid == 0) p.chunk_start[0] = 0;
    return;
  }
  const int per_layer = p.B * p.H_kv;
  for (int base = 0; base < u1; base += blockDim.x) {
    const int u = base + tid;
    int c = 0, n = 0;
    if (u < p.n_units) {
      const int ls = u / per_layer;
      const int s = (u - ls * per_layer) / p.H_kv;
      n = p.lens_in[s];
      if (n < 0 || n > p.S_cap) n = 0;  // flagged by CTA 0
      const bool h2o = p.slayer_method[ls] == KVEV_H2O;
      // H2O layers scored over the whole prompt have their own kernels
      const bool need =
          n > 0 && !p.slayer_ext[ls] && (h2o ? p.mode != kScoreNoH2O : n > p.slayer_budget[ls]);
      c = need ? (n + p.chunk_keys - 1) / p.chunk_keys : 0;
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
    if (u >= u0 && u < u1) {
      p.chunk_start[u] = excl;
      p.ready[u] = 0;
      if ((excl + c) * kTreeLevels > p.n_node_cnt) {  // never for a workspace of ws_layout's size
        atomicOr(p.status, kStatusDevice);
        c = 0;
      }
      for (int q = 0; q < c; ++q) {
        const int key0 = q * p.chunk_keys;
        const int nk = min(p.chunk_keys, n - key0);
        const int ntiles = (nk + kTileKeys - 1) / kTileKeys;
        p.item[excl + q] = make_int4(u, n, key0, ntiles | (c << 16));
#pragma unroll
        for (int lv = 0; lv < kTreeLevels; ++lv) p.node_cnt[(excl + q) * kTreeLevels + lv] = 0;
      }
    }
    __syncthreads();
    if (tid == blockDim.x - 1) carry = excl + c;
    __syncthreads();
  }
  if (u1 == p.n_units && tid == 0) p.chunk_start[p.n_units] = carry;
}

// ---------------------------------------------------------------------------
// Supplied normalisers: the caller's log-sum-exp of every window row (the
// softmax_lse of its own prefill attention), as -base-2 values in each
// scored unit's normaliser row, the unit then marked ready.  One CTA per
// scoring unit; rows that lie before the sequence start get +inf (no key
// sees them).  Runs after the prologue, which clears the ready flags.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) lse_fill_kernel(const __grid_constant__ LseParams p) {
  const int u = blockIdx.x;
  const int per_layer = p.B * p.H_kv;
  const int ls = u / per_layer;
  const int rem = u - ls * per_layer;
  const int s = rem / p.H_kv, h = rem - s * p.H_kv;
  const int n = p.lens[s];
  const float* lse = p.lse[ls];
  if (lse == nullptr) return;  // a layer whose scores the caller supplies
  constexpr float kInvLn2 = 1.4426950408889634f;
  for (int r = threadIdx.x; r < p.R_pad; r += blockDim.x) {
    const int g = r / p.W, i = r - g * p.W;
    const bool valid = r < p.R && n - p.W + i >= 0;
    p.lam[static_cast<size_t>(u) * p.R_pad + r] =
        valid ? lse[(static_cast<size_t>(s) * p.H_q + h * p.G + g) * p.W + i] * kInvLn2 : INFINITY;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) st_release(&p.ready[u], 1);
}

}  // namespace

cudaError_t launch_lse_fill(const LseParams& p, cudaStream_t s) {
  if (p.n_units == 0) return cudaSuccess;
  lse_fill_kernel<<<p.n_units, 256, 0, s>>>(p);
  return cudaGetLastError();
}

int score_smem_bytes(int d, int q_rows, int q_bufs, int R_pad, int stages) {
  size_t koff, loff, roff, poff, boff;
  const size_t off = smem_size(d, q_rows, q_bufs, R_pad, stages, &koff, &loff, &roff, &poff, &boff);
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
  // about 128 units per CTA
  const int want = (p.n_units + 127) / 128;
  const int grid = want < 1 ? 1 : want > 256 ? 256 : want;
  prologue_kernel<<<grid, 1024, 0, s>>>(p);
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
