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
// Roles per CTA (320 threads): warp 0 issues TMA loads (one thread), warp 1
// owns TMEM and issues tcgen05.mma (one thread), warps 2-5 and 6-9 are two
// softmax warpgroups that take alternate tiles, each with its own TMEM
// accumulator buffer.
#include "kvev_internal.cuh"

namespace kvev {

namespace {

struct Smem {
  uint8_t* qbuf;     // two Q buffers of qbytes each, indexed arithmetically (a dynamically
  uint32_t qbytes;   // indexed member array would push the whole struct to local memory)
  uint8_t* kbuf;     // stages * tile bytes
  float* lam[2];     // per warpgroup copy of lse2 of the current sweep-2 unit
  uint64_t* kfull;
  uint64_t* kempty;
  uint64_t* qfull;
  uint64_t* qempty;
  uint64_t* tfull;
  uint64_t* tempty;
  uint64_t* done;
  uint32_t* tmem_slot;
  int* flag;         // [4]: [wg] last-arrival of sweep 1, [2+wg] ready of sweep 2
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
  s.lam[0] = reinterpret_cast<float*>(base + off);
  off += sizeof(float) * p.R_pad;
  s.lam[1] = reinterpret_cast<float*>(base + off);
  off += sizeof(float) * p.R_pad;
  off = (off + 7) & ~size_t(7);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + off);
  s.kfull = bars;
  s.kempty = bars + p.stages;
  s.qfull = bars + 2 * p.stages;
  s.qempty = s.qfull + 2;
  s.tfull = s.qempty + 2;
  s.tempty = s.tfull + 2;
  s.done = s.tempty + 2;
  s.tmem_slot = reinterpret_cast<uint32_t*>(s.done + 1);
  s.flag = reinterpret_cast<int*>(s.tmem_slot + 1);
  return s;
}

struct ItemInfo {
  int u, s, h, ls, n, key0, ntiles, cs, nchunks;
};

__device__ __forceinline__ ItemInfo item_info(const ScoreParams& p, int t) {
  ItemInfo it;
  it.u = p.item_unit[t];
  it.cs = p.chunk_start[it.u];
  it.nchunks = p.chunk_start[it.u + 1] - it.cs;
  const int per_layer = p.B * p.H_kv;
  it.ls = it.u / per_layer;
  const int rem = it.u - it.ls * per_layer;
  it.s = rem / p.H_kv;
  it.h = rem - it.s * p.H_kv;
  it.n = p.lens[it.s];
  const int c = t - it.cs;
  it.key0 = c * p.chunk_keys;
  int nk = it.n - it.key0;
  if (nk > p.chunk_keys) nk = p.chunk_keys;
  it.ntiles = (nk + kTileKeys - 1) / kTileKeys;
  return it;
}

// Bounded wait on an mbarrier phase; false if it ran out or another role aborted.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, const ScoreParams& p) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  uint32_t spins = 0;
  while (!mbar_try_wait(bar, parity)) {
    if ((++spins & 63u) == 0) {
      if (ld_volatile(p.abort_flag)) return false;
      if (globaltimer_ns() - t0 > static_cast<uint64_t>(p.wait_ns)) {
        atomicExch(p.abort_flag, 1);
        atomicOr(p.status, kStatusTimeout);
        return false;
      }
    }
  }
  return true;
}

// Bounded wait used while shutting down: ignores the abort flag, gives up after
// `ns` nanoseconds (asynchronous copies and MMAs finish on their own).
__device__ __forceinline__ void wait_bar_drain(uint64_t* bar, uint32_t parity, uint64_t ns) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > ns) return;
}

// ---------------------------------------------------------------------------
// Producer: TMA loads of Q (once per item) and of K tiles (twice per item).
// ---------------------------------------------------------------------------
template <int D>
__device__ void producer(const ScoreParams& p, const Smem& sm, int first, int stride, int J) {
  constexpr uint32_t kTileBytes = kTileKeys * D * 2;
  const uint32_t qbytes = static_cast<uint32_t>(p.R_pad) * D * 2;
  const uint64_t keep = policy_evict_last();   // first read of a K tile: keep it for the re-read
  const uint64_t drop = policy_evict_first();  // second read: its last use
  uint32_t tile = 0;
  int last_q_item = -1;
  int issued_q0 = 0, issued_q1 = 0;  // Q loads issued into each buffer
  bool ok = true;
  for (int j = 0; j <= J && ok; ++j) {
    for (int sweep = 0; sweep < 2 && ok; ++sweep) {
      const int jj = sweep == 0 ? j : j - 1;
      if (sweep == 0 && j >= J) continue;
      if (sweep == 1 && j == 0) continue;
      const int t = first + jj * stride;
      const ItemInfo it = item_info(p, t);
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
        const uint32_t st = tile % p.stages;
        const uint32_t ph = (tile / p.stages) & 1;
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
// MMA issuer (one thread): sweep 1 -> S = Q K^T, sweep 2 -> S^T = K Q^T.
// ---------------------------------------------------------------------------
template <int D>
__device__ void mma_issuer(const ScoreParams& p, const Smem& sm, uint32_t tmem_base, int first,
                           int stride, int J) {
  constexpr uint32_t kTileBytes = kTileKeys * D * 2;
  const int nh = p.R_pad > 128 ? 2 : 1;
  const uint32_t idesc1 = idesc_bf16_f32(128, kTileKeys);
  const uint32_t idesc2 = idesc_bf16_f32(128, p.R_pad);
  const uint32_t qcol_bytes = static_cast<uint32_t>(p.q_rows) * 128;  // one 64-wide column block
  uint32_t tile = 0;
  bool ok = true;
  for (int j = 0; j <= J && ok; ++j) {
    for (int sweep = 0; sweep < 2 && ok; ++sweep) {
      const int jj = sweep == 0 ? j : j - 1;
      if (sweep == 0 && j >= J) continue;
      if (sweep == 1 && j == 0) continue;
      const int t = first + jj * stride;
      const ItemInfo it = item_info(p, t);
      const int qb = jj & 1;
      const uint32_t qaddr = smem_u32(sm.qbuf) + qb * sm.qbytes;
      if (sweep == 0) {
        if (!wait_bar(&sm.qfull[qb], (jj >> 1) & 1, p)) { ok = false; break; }
      }
      for (int i = 0; i < it.ntiles; ++i, ++tile) {
        const uint32_t st = tile % p.stages;
        const uint32_t buf = tile & 1;
        if (!wait_bar(&sm.kfull[st], (tile / p.stages) & 1, p)) { ok = false; break; }
        if (!wait_bar(&sm.tempty[buf], ((tile >> 1) & 1) ^ 1, p)) { ok = false; break; }
        tc_fence_after();
        const uint32_t kaddr = smem_u32(sm.kbuf) + st * kTileBytes;
        const uint32_t dcol = tmem_base + buf * p.tmem_buf_cols;
        if (sweep == 0) {
          for (int h = 0; h < nh; ++h) {
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
              const uint32_t koff = (k >> 2) * (kTileKeys * 128) + (k & 3) * 32;
              const uint32_t qoff = (k >> 2) * qcol_bytes + h * (128 * 128) + (k & 3) * 32;
              umma_bf16(dcol + h * 128, sw128_desc(qaddr + qoff), sw128_desc(kaddr + koff),
                        idesc1, k > 0);
            }
          }
        } else {
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {
            const uint32_t koff = (k >> 2) * (kTileKeys * 128) + (k & 3) * 32;
            const uint32_t qoff = (k >> 2) * qcol_bytes + (k & 3) * 32;
            umma_bf16(dcol, sw128_desc(kaddr + koff), sw128_desc(qaddr + qoff), idesc2, k > 0);
          }
        }
        umma_commit(&sm.kempty[st]);
        umma_commit(&sm.tfull[buf]);
      }
      if (ok && sweep == 1) umma_commit(&sm.qempty[qb]);
    }
  }
  // Every MMA issued so far has completed once `done` flips.
  umma_commit(sm.done);
  wait_bar_drain(sm.done, 0, 1000000000ull);
}

// ---------------------------------------------------------------------------
// Softmax warpgroups.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int row_pos(const ScoreParams& p, int r, int n) {
  // absolute position of window row r; < 0 means the row lies before the sequence
  return n - p.W + (r % p.W);
}

// Sweep 1 on one tile: update the running base-2 (max, sum) of the rows this
// thread owns (row lrow of each 128-row half).
__device__ __forceinline__ void sweep1_tile(const ScoreParams& p, uint32_t taddr, int lrow,
                                            int nh, int n, int kb, float (&m)[2], float (&z)[2]) {
  const float c = p.scale_log2;
  for (int h = 0; h < 2; ++h) {
    if (h >= nh) break;
    const int r = h * 128 + lrow;
    const bool row_ok = r < p.R;
    const int tr = row_ok ? row_pos(p, r, n) : -1;
    const bool full = (kb + kTileKeys - 1) <= (n - p.W);  // every key visible to every row
#pragma unroll 1
    for (int c0 = 0; c0 < kTileKeys; c0 += 32) {
      float v[32];
      tmem_ld32(taddr + h * 128 + c0, v);
      if (!row_ok || tr < 0) continue;
      float vmax = -INFINITY;
      if (full) {
#pragma unroll
        for (int i = 0; i < 32; ++i) vmax = fmaxf(vmax, v[i]);
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          if (kb + c0 + i > tr) v[i] = -INFINITY;
          vmax = fmaxf(vmax, v[i]);
        }
      }
      if (vmax == -INFINITY) continue;
      const float mnew = fmaxf(m[h], vmax * c);
      float zz = z[h] * ex2_approx(m[h] - mnew);  // m = -inf -> 0
      float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        acc0 += ex2_approx(fmaf(v[i], c, -mnew));
        acc1 += ex2_approx(fmaf(v[i + 1], c, -mnew));
      }
      z[h] = zz + (acc0 + acc1);
      m[h] = mnew;
    }
  }
}

// Sweep 2 on one tile: this thread's key kb + lrow against all R rows.
__device__ __forceinline__ void sweep2_tile(const ScoreParams& p, uint32_t taddr, int lrow, int n,
                                            int kb, const float* lam, float* raw_unit) {
  const float c = p.scale_log2;
  const int k = kb + lrow;
  const bool key_ok = k < n;
  const bool full = (kb + kTileKeys - 1) < (n - p.W);  // every row sees every key of the tile
  float acc0 = 0.f, acc1 = 0.f;
  int c0 = 0;
#pragma unroll 1
  for (; c0 + 32 <= p.R_pad; c0 += 32) {
    float v[32];
    tmem_ld32(taddr + c0, v);
    if (!key_ok) continue;
    if (full && c0 + 32 <= p.R) {
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        acc0 += ex2_approx(fmaf(v[i], c, -lam[c0 + i]));
        acc1 += ex2_approx(fmaf(v[i + 1], c, -lam[c0 + i + 1]));
      }
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int r = c0 + i;
        if (r < p.R && k <= row_pos(p, r, n)) acc0 += ex2_approx(fmaf(v[i], c, -lam[r]));
      }
    }
  }
  if (c0 < p.R_pad) {  // a 16-column tail
    float v[16];
    tmem_ld16(taddr + c0, v);
    if (key_ok) {
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int r = c0 + i;
        if (r < p.R && k <= row_pos(p, r, n)) acc0 += ex2_approx(fmaf(v[i], c, -lam[r]));
      }
    }
  }
  if (key_ok) raw_unit[k] = (acc0 + acc1) * p.inv_G;
}

__device__ void softmax_wg(const ScoreParams& p, const Smem& sm, uint32_t tmem_base, int wg,
                           int first, int stride, int J) {
  const int warp = threadIdx.x >> 5;
  const int quarter = warp & 3;           // TMEM lane quarter this warp may access
  const int lrow = quarter * 32 + (threadIdx.x & 31);
  const int wtid = threadIdx.x - (2 + 4 * wg) * 32;  // 0..127 within the warpgroup
  const int bar_id = 1 + wg;
  const int nh = p.R_pad > 128 ? 2 : 1;
  const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16);
  float* lam_s = sm.lam[wg];
  uint32_t tile = 0;
  bool ok = true;

  for (int j = 0; j <= J; ++j) {
    // ---------------- sweep 1 of item j ----------------
    if (j < J) {
      const int t = first + j * stride;
      const ItemInfo it = item_info(p, t);
      float m[2] = {-INFINITY, -INFINITY}, z[2] = {0.f, 0.f};
      for (int i = 0; i < it.ntiles; ++i) {
        const uint32_t gt = tile + i;
        if ((gt & 1) != static_cast<uint32_t>(wg)) continue;
        if (ok && !wait_bar(&sm.tfull[wg], (gt >> 1) & 1, p)) ok = false;
        ok = __all_sync(0xffffffffu, ok);  // tcgen05.ld needs the whole warp
        if (ok) {
          tc_fence_after();
          sweep1_tile(p, lane_addr + wg * p.tmem_buf_cols, lrow, nh, it.n,
                      it.key0 + i * kTileKeys, m, z);
        }
        tc_fence_before();
        mbar_arrive(&sm.tempty[wg]);
      }
      tile += it.ntiles;
      // publish this warpgroup's partial of the chunk
      float2* part = p.part + (static_cast<size_t>(t) * 2 + wg) * p.R_pad;
      for (int h = 0; h < nh; ++h) {
        const int r = h * 128 + lrow;
        if (r < p.R_pad) part[r] = make_float2(m[h], z[h]);
      }
      __threadfence();
      named_bar_sync(bar_id, 128);
      if (wtid == 0) {
        const int old = atomicAdd(&p.cnt[it.u], 1);
        __threadfence();
        sm.flag[wg] = (old == 2 * it.nchunks - 1);
      }
      named_bar_sync(bar_id, 128);
      if (sm.flag[wg]) {
        // Last arrival for this unit: merge every chunk's (max, sum) partials
        // of each row into lse2 = M + log2(Z) in one pass, with eight
        // independent loads in flight (this runs while the unit's other
        // chunk-holders wait for it).
        for (int h = 0; h < nh; ++h) {
          const int r = h * 128 + lrow;
          if (r >= p.R_pad) continue;
          const float2* pp = p.part + static_cast<size_t>(it.cs) * 2 * p.R_pad + r;
          const int nq = 2 * it.nchunks;
          float M = -INFINITY, Z = 0.f;
          for (int q0 = 0; q0 < nq; q0 += 8) {
            float2 e[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
              e[i] = q0 + i < nq ? __ldcg(&pp[static_cast<size_t>(q0 + i) * p.R_pad])
                                 : make_float2(-INFINITY, 0.f);
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
      const ItemInfo it = item_info(p, t);
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
        sm.flag[2 + wg] = ready;
      }
      named_bar_sync(bar_id, 128);
      const bool have = sm.flag[2 + wg] != 0;
      for (int r = wtid; r < p.R_pad; r += 128)
        lam_s[r] = have ? __ldcg(&p.lam[static_cast<size_t>(it.u) * p.R_pad + r]) : INFINITY;
      named_bar_sync(bar_id, 128);
      float* raw_unit = p.raw + static_cast<size_t>(it.u) * p.S_cap;
      for (int i = 0; i < it.ntiles; ++i) {
        const uint32_t gt = tile + i;
        if ((gt & 1) != static_cast<uint32_t>(wg)) continue;
        if (ok && !wait_bar(&sm.tfull[wg], (gt >> 1) & 1, p)) ok = false;
        ok = __all_sync(0xffffffffu, ok);
        if (ok) {
          tc_fence_after();
          sweep2_tile(p, lane_addr + wg * p.tmem_buf_cols, lrow, it.n, it.key0 + i * kTileKeys,
                      lam_s, raw_unit);
        }
        tc_fence_before();
        mbar_arrive(&sm.tempty[wg]);
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
      mbar_init(&sm.tfull[i], 1);
      mbar_init(&sm.tempty[i], 128);
    }
    mbar_init(sm.done, 1);
    fence_barrier_init();
    fence_proxy_async();
  }
  if (warp == 1) {
    tmem_alloc(sm.tmem_slot, 2 * p.tmem_buf_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *sm.tmem_slot;

  const int total = p.chunk_start[p.n_units];
  const int first = blockIdx.x, stride = gridDim.x;
  const int J = first < total ? (total - first + stride - 1) / stride : 0;

  if (warp == 0) {
    if ((threadIdx.x & 31) == 0) producer<D>(p, sm, first, stride, J);
  } else if (warp == 1) {
    if ((threadIdx.x & 31) == 0) mma_issuer<D>(p, sm, tmem_base, first, stride, J);
  } else {
    softmax_wg(p, sm, tmem_base, (warp - 2) >> 2, first, stride, J);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 2 * p.tmem_buf_cols);
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
      for (int q = 0; q < c; ++q) p.item_unit[excl + q] = u;
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
  off += 2 * sizeof(float) * R_pad;
  off = (off + 7) & ~size_t(7);
  off += sizeof(uint64_t) * (2 * stages + 9);
  off += sizeof(uint32_t) + 4 * sizeof(int);
  return static_cast<int>((off + 127) & ~size_t(127));
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
