// kvev_internal.cuh -- device helpers and launch parameter blocks shared by the
// kernels of libkvev.so (GB300 / sm_103a).  Inline PTX for mbarrier, TMA and
// the 5th-generation tensor core (tcgen05 + tensor memory).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvev.h"

namespace kvev {

constexpr int kMaxLayers = 128;       // layers in one plan
constexpr int kMaxScoreLayers = 64;   // SnapKV/H2O layers (tensor maps travel as kernel params)
constexpr int kTileKeys = 128;        // keys per tensor-core tile (MMA M or N)
constexpr int kSuperKeys = 256;       // keys per K stage (sweep 1 MMAs take N = 256 keys)
// Tiles per scoring work item (chunk), at least.  Larger chunks give each CTA
// more slack before it needs a unit's normaliser and halve the partials to
// merge; the cost is reuse distance (grid * chunk bytes between a tile's two
// reads, ~78 MB at 16 tiles on 152 SMs, inside the 126 MB L2).
constexpr int kMinChunkTiles = 16;
// The per-row (max, sum) records of a unit's chunks are merged up a tree of
// fan-in kTreeFanIn (the last child to arrive merges its siblings), so the
// normaliser is ready a few load round trips after the unit's last chunk.
// What a prologue + score launch covers (PrologueParams::mode).
constexpr int kScoreAll = 0;       // every scoring layer, rows = the observation window
constexpr int kScoreNoH2O = 1;     // SnapKV layers only (H2O layers are scored over the whole prompt)
constexpr int kTreeFanIn = 4;
constexpr int kTreeLevels = 5;        // internal levels: up to 4^5 = 1024 chunks per unit
constexpr int kSoftmaxWGs = 4;        // softmax warpgroups of the score kernel
constexpr int kRedTiles = 8;          // sweep-2 tiles whose key sums are combined at once
constexpr int kScoreThreads = 128 * (1 + kSoftmaxWGs);  // + warpgroup 0: TMA, MMA, publisher, normaliser warps
constexpr int kSlots = 4;             // TMEM accumulator slots of the score kernel
constexpr int kSlotCols = 128;        // fp32 columns per slot (4 x 128 = all 512 columns)
// Register split of the score kernel (setmaxnreg): warpgroup 0 shrinks to 64,
// the softmax warpgroups grow to 104.  The CTA must be launched with at least
// 128 * 64 + 512 * 104 = 61440 registers (96 per thread x 640): the host
// checks the compiled allocation before launching, since an increase that the
// launch pool cannot cover would never complete.
constexpr int kRegsControl = 64;
constexpr int kRegsSoftmax = 104;
constexpr int kRegsNeeded = 128 * kRegsControl + 128 * kSoftmaxWGs * kRegsSoftmax;
constexpr int kSelectThreads = 256;    // one selection CTA per unit
constexpr int kSelectCtasPerSm = 4;    // resident selection CTAs an SM should hold
constexpr int kWsAlign = 256;

// Bits of the device status word.
constexpr int kStatusTimeout = 1;
constexpr int kStatusDevice = 2;

// Per-layer description used by the selection and gather kernels.
struct LayerDesc {
  int method;         // prefill operator (KVEV_*)
  int slots;          // output slots per (seq, kv head): b_l, 0 for FULL
  int recent;         // StreamingLLM recent tokens kept (<= b - sink)
  int h2o_recent;     // H2O protected recent window
  int score_slot;     // index among scoring layers, -1 if none
  long long row_off;  // first packed output row of the layer
  const float* scores;  // [B*H_kv][S_cap] scores of a scoring layer: its workspace slot, or the
                        // caller's array when the caller supplies them; null otherwise
};

struct PrologueParams {
  int n_units;        // scoring units = n_slayers * B * H_kv
  int B, H_kv, S_cap;
  int chunk_keys;
  int slayer_method[kMaxScoreLayers];
  int slayer_budget[kMaxScoreLayers];
  int slayer_ext[kMaxScoreLayers];  // 1: the caller supplies the layer's scores (not scored here)
  const int* lens_in; // caller's lengths
  int* lens;          // validated copy (out-of-range lengths become 0, flagged)
  int* status;
  int* node_cnt;      // [items][kTreeLevels] arrival counters of the merge tree (zeroed here)
  int n_node_cnt;     // counters in node_cnt (workspace capacity)
  int W;              // observation window
  int mode;           // kScoreAll, or kScoreNoH2O (H2O layers are scored over the whole prompt)
  int* ready;
  int* abort_flag;
  int* chunk_start;   // [n_units + 1]
  int4* item;         // [items] {unit, n, first key, tiles | chunks of the unit << 16}
};

struct ScoreParams {
  CUtensorMap kmap[kMaxScoreLayers];  // K of each scoring layer, 2-D {d, B*H_kv*S_cap}
  CUtensorMap qmap[kMaxScoreLayers];  // Q_win of each scoring layer, 2-D {d, B*H_q*W}
  int n_units, B, H_kv, H_q, G, W, R, R_pad, S_cap;
  int chunk_keys;     // keys per work item (multiple of 128)
  int q_rows;         // rows of a Q shared-memory buffer (128 or 256)
  int q_bufs;         // Q buffers (2: the next entry's Q loads during this entry; 1: it
                      // loads once this entry is done, leaving room for more K stages)
  int stages;         // K tile ring depth
  float scale_log2;   // log2(e) / sqrt(d)
  float inv_G;
  const int* lens;
  const int* chunk_start;
  const int4* item;   // [items] {unit, n, first key, tiles | chunks of the unit << 16}
  int* node_cnt;      // [items][kTreeLevels]: counter of the tree node whose first leaf is the item
  int* ready;
  int* abort_flag;
  int* status;
  float2* part;       // [items][R_pad] per-row (max, sum) of a chunk, or of the tree node
                      // whose first leaf is that chunk, base-2 units
  float* lam;         // [n_units][R_pad] per-row log2-sum-exp
  float* raw;         // [n_units][S_cap] window scores
  long long wait_ns;
  int stall_unit;
  int single;         // 1: the normalisers are supplied (lse_fill_kernel); sweep 2 only
  // ---- whole-prompt H2O scoring (h2o_full.cu) ----
  int phase;          // 0: row pass (lse2 of every prompt row), 1: key pass (scores)
  int Pb;             // prompt positions per query block (G * Pb <= 256 rows)
  int n_h2o;          // H2O scoring layers
  int h2o_slot[kMaxScoreLayers];  // their scoring-layer indices
  int nb_max;         // query blocks of a full-capacity unit: ceil(S_cap / Pb)
  int nkt_max;        // 256-key super-tiles of a full-capacity unit
  int n_items;        // items of the pass: (nb_max or nkt_max) x H2O units
  float* lse;         // [H2O unit][G][S_cap] base-2 log-sum-exp of every prompt row
  const float* lse_src[kMaxScoreLayers];  // the caller's every-row log-sum-exp per H2O layer
                      // (fp32 [B][H_q][S_cap], natural log), or null: the row pass computes it
};

// The caller's window-row log-sum-exp (natural log, softmax scale included)
// of each scoring layer, fp32 [B][H_q][W], into the units' normaliser rows.
struct LseParams {
  const float* lse[kMaxScoreLayers];  // null: the layer's scores are supplied instead
  int n_units, B, H_kv, H_q, G, W, R, R_pad;
  const int* lens;
  float* lam;         // [n_units][R_pad] lse2 of the rows (+inf: no row)
  int* ready;
};

struct SelectParams {
  LayerDesc layer[kMaxLayers];
  int order[kMaxLayers];  // layers in dispatch order: the L_first scoring layers, then the rest
  int L_first;
  int L, B, H_kv, S_cap, W, pool_kernel, pool_type, sink, d;
  const int* lens;
  int* out_idx;
  int* out_count;     // [L][B][H_kv]
  uint32_t* keys;     // workspace: [scoring unit][key_stride] selection keys
  int key_stride;     // S_cap rounded up to a multiple of 128 (whole transposed key blocks)
  // StreamingLLM layers: their kept rows are copied by the selection launch
  const void* K[kMaxLayers];
  const void* V[kMaxLayers];
  void* out_K;
  void* out_V;
};

// Per-layer description of the decode arena.
struct DecLayer {
  int method;         // decode-phase operator (KVEV_*); FULL = append only
  int b;              // budget: slots kept by an evicting layer
  int cap;            // slots per unit in the arena (0: the layer has no arena)
  int r;              // H2O / TOVA protected recent window
  int sink, recent;   // StreamingLLM
  int pre_method;     // prefill operator (its packed rows seed the arena)
  int pre_slots;      // prefill slots per unit (b_l)
  int unit_off;       // first unit of the layer
  int att_end;        // H2O / TOVA units of layers 0..l (one CTA each in the step kernel)
  int cheap_end;      // StreamingLLM and append-only units of layers 0..l (one warp each)
  long long row_off;  // first arena slot row of the layer
  long long pre_row_off;  // first packed prefill row of the layer
};

struct DecodeParams {
  DecLayer layer[kMaxLayers];
  const void* k_new[kMaxLayers];  // [B][H_kv][d] bf16 per layer
  const void* v_new[kMaxLayers];  // [B][H_kv][d]
  const void* q_new[kMaxLayers];  // [B][H_q][d]
  const float* attn[kMaxLayers];  // [B][H_kv][cap + 1] caller-supplied attention, or null
  int L, B, H_kv, H_q, G, d, units;
  int n_att, n_cheap; // attending units; StreamingLLM and append-only units
  float scale_log2;   // log2(e) / sqrt(d)
  void* K;            // arena rows [rows][d] bf16
  void* V;
  int32_t* pos;       // [rows]
  float* acc;         // [rows]
  int32_t* count;     // [units]
  int32_t* evicted;   // [units]: position evicted by the last step, -1 = none
  int32_t* lens;      // [B]
  int32_t* done;      // units finished in the current step; the last one advances lens
  int* status;
  // initialisation from the packed prefill output
  const void* pre_K;
  const void* pre_V;
  const int32_t* pre_idx;
  const int32_t* pre_count;  // [L][B][H_kv]
  const float* h2o_state;    // nullable
  const int32_t* lens_in;    // [B]
};

struct GatherParams {
  LayerDesc layer[kMaxLayers];
  const void* K[kMaxLayers];
  const void* V[kMaxLayers];
  long long grow_off[kMaxLayers];  // first gathered row of the layer (SnapKV / H2O layers own rows)
  int L, B, H_kv, S_cap, d;
  long long total_rows;  // gathered rows: the packed rows of the SnapKV and H2O layers
  const int* out_idx;
  void* out_K;
  void* out_V;
  float* h2o_state;
  int* status;
};

// ---------------------------------------------------------------------------
// Small PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// mbarrier arrive from the lane that elect.sync picks in a converged warp.
__device__ __forceinline__ void mbar_arrive_elect(uint64_t* bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e mbarrier.arrive.shared::cta.b64 _, [%0];\n\t}" ::"r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait with a suspend-time hint: the thread sleeps in hardware until the
// phase completes or about `hint_ns` pass, instead of polling (polling warps
// take issue slots from the warps doing the work).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 2-D tiled TMA load into shared memory, completion counted on `bar`.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Same, with an L2 cache-eviction policy (from createpolicy).
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_load_2d_hint(void* dst, const CUtensorMap* map, int x, int y,
                                                 uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---- tcgen05 -----------------------------------------------------------------

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D(tmem) (+)= A(smem) * B(smem)^T, bf16 inputs, fp32 accumulate, one CTA.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// The same MMA issued from a whole converged warp: one elected lane issues, so
// the warp-uniform operands can stay in uniform registers.
__device__ __forceinline__ void umma_bf16_elect(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p, e;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// tcgen05.commit from the lane that elect.sync picks in a converged warp (the
// same lane that issued the MMAs through umma_bf16_elect).
__device__ __forceinline__ void umma_commit_elect(uint64_t* bar) {
  asm volatile(
      "{\n\t.reg .pred e;\n\t"
      "elect.sync _|e, 0xffffffff;\n\t"
      "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(
          smem_u32(bar))
      : "memory");
}

// Arrive on `bar` once every tcgen05 operation issued so far by this thread completes.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Issue a load of 32 consecutive fp32 columns of this thread's TMEM lane; the
// registers are valid only after tmem_wait32() on the same array.
// 64 consecutive fp32 columns of this thread's TMEM lane in one load: columns
// [0, 32) into r0 and [32, 64) into r1; valid only after tmem_wait64().
__device__ __forceinline__ void tmem_ld64_async(uint32_t taddr, uint32_t (&r0)[32], uint32_t (&r1)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];"
      : "=r"(r0[0]), "=r"(r0[1]), "=r"(r0[2]), "=r"(r0[3]), "=r"(r0[4]), "=r"(r0[5]), "=r"(r0[6]), "=r"(r0[7]), "=r"(r0[8]), "=r"(r0[9]), "=r"(r0[10]), "=r"(r0[11]), "=r"(r0[12]), "=r"(r0[13]), "=r"(r0[14]), "=r"(r0[15]), "=r"(r0[16]), "=r"(r0[17]), "=r"(r0[18]), "=r"(r0[19]), "=r"(r0[20]), "=r"(r0[21]), "=r"(r0[22]), "=r"(r0[23]), "=r"(r0[24]), "=r"(r0[25]), "=r"(r0[26]), "=r"(r0[27]), "=r"(r0[28]), "=r"(r0[29]), "=r"(r0[30]), "=r"(r0[31]), "=r"(r1[0]), "=r"(r1[1]), "=r"(r1[2]), "=r"(r1[3]), "=r"(r1[4]), "=r"(r1[5]), "=r"(r1[6]), "=r"(r1[7]), "=r"(r1[8]), "=r"(r1[9]), "=r"(r1[10]), "=r"(r1[11]), "=r"(r1[12]), "=r"(r1[13]), "=r"(r1[14]), "=r"(r1[15]), "=r"(r1[16]), "=r"(r1[17]), "=r"(r1[18]), "=r"(r1[19]), "=r"(r1[20]), "=r"(r1[21]), "=r"(r1[22]), "=r"(r1[23]), "=r"(r1[24]), "=r"(r1[25]), "=r"(r1[26]), "=r"(r1[27]), "=r"(r1[28]), "=r"(r1[29]), "=r"(r1[30]), "=r"(r1[31])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait64(uint32_t (&r0)[32], uint32_t (&r1)[32]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(r0[0]), "+r"(r0[1]), "+r"(r0[2]), "+r"(r0[3]), "+r"(r0[4]), "+r"(r0[5]), "+r"(r0[6]), "+r"(r0[7]), "+r"(r0[8]), "+r"(r0[9]), "+r"(r0[10]), "+r"(r0[11]), "+r"(r0[12]), "+r"(r0[13]), "+r"(r0[14]), "+r"(r0[15]), "+r"(r0[16]), "+r"(r0[17]), "+r"(r0[18]), "+r"(r0[19]), "+r"(r0[20]), "+r"(r0[21]), "+r"(r0[22]), "+r"(r0[23]), "+r"(r0[24]), "+r"(r0[25]), "+r"(r0[26]), "+r"(r0[27]), "+r"(r0[28]), "+r"(r0[29]), "+r"(r0[30]), "+r"(r0[31]), "+r"(r1[0]), "+r"(r1[1]), "+r"(r1[2]), "+r"(r1[3]), "+r"(r1[4]), "+r"(r1[5]), "+r"(r1[6]), "+r"(r1[7]), "+r"(r1[8]), "+r"(r1[9]), "+r"(r1[10]), "+r"(r1[11]), "+r"(r1[12]), "+r"(r1[13]), "+r"(r1[14]), "+r"(r1[15]), "+r"(r1[16]), "+r"(r1[17]), "+r"(r1[18]), "+r"(r1[19]), "+r"(r1[20]), "+r"(r1[21]), "+r"(r1[22]), "+r"(r1[23]), "+r"(r1[24]), "+r"(r1[25]), "+r"(r1[26]), "+r"(r1[27]), "+r"(r1[28]), "+r"(r1[29]), "+r"(r1[30]), "+r"(r1[31])
      :
      : "memory");
}

__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}

// Wait for every outstanding TMEM load.  The array is tied to the wait as an
// in/out operand so no use of its registers can be scheduled before it.
__device__ __forceinline__ void tmem_wait32(uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
        "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]),
        "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]),
        "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]),
        "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]),
        "+r"(r[31])
      :
      : "memory");
}

// Two-lane packed fp32 fused multiply-add (one instruction for two values).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  uint64_t ra, rb, rc, rd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rc) : "f"(c.x), "f"(c.y));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(rd) : "l"(ra), "l"(rb), "l"(rc));
  float2 d;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
  return d;
}

// Two-lane packed fp32 add.
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  uint64_t ra, rb, rd;
  asm("mov.b64 %0, {%1, %2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1, %2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(rd) : "l"(ra), "l"(rb));
  float2 d;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
  return d;
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ float4 lds4(const float* p) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(smem_u32(p)));
  return v;
}

__device__ __forceinline__ float lds1(const float* p) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(smem_u32(p)));
  return v;
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  tmem_wait_ld();
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  tmem_wait_ld();
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor of a K-major bf16 operand stored with the
// 128-byte swizzle: rows of 128 B (64 elements), 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);  // start address
  d |= static_cast<uint64_t>(16u >> 4) << 16;           // leading-dim byte offset (unused)
  d |= static_cast<uint64_t>(1024u >> 4) << 32;         // stride between 8-row groups
  d |= static_cast<uint64_t>(1) << 46;                  // descriptor version
  d |= static_cast<uint64_t>(2) << 61;                  // 128-byte swizzle
  return d;
}

// Instruction descriptor: kind::f16 with bf16 A/B, fp32 D, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int N>
__device__ __forceinline__ void regs_dealloc() {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
template <int N>
__device__ __forceinline__ void regs_alloc() {
  asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int ld_volatile(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}

// Order-preserving map of an fp32 to uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t float_key(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

}  // namespace kvev

// Launchers implemented by the kernel translation units.
namespace kvev {
cudaError_t launch_prologue(const PrologueParams& p, cudaStream_t s);
cudaError_t launch_score(const ScoreParams& p, int d, int grid, size_t smem, cudaStream_t s);
int score_smem_bytes(int d, int q_rows, int q_bufs, int R_pad, int stages);
bool decode_supported(int d, int G);
cudaError_t launch_decode_init(const DecodeParams& p, cudaStream_t s);
cudaError_t launch_decode_step(const DecodeParams& p, size_t smem, cudaStream_t s);
int score_kernel_regs(int d);
cudaError_t score_set_smem(int d, size_t smem);
int h2o_full_smem_bytes(int d);
int h2o_full_kernel_regs(int d);
cudaError_t h2o_full_set_smem(int d, size_t smem);
cudaError_t launch_h2o_full(const ScoreParams& p, int d, int grid, size_t smem, cudaStream_t s);
cudaError_t launch_lse_fill(const LseParams& p, cudaStream_t s);
cudaError_t launch_lse_rows_fill(const ScoreParams& p, cudaStream_t s);
cudaError_t launch_select(const SelectParams& p, int grid, cudaStream_t s);
cudaError_t launch_gather(const GatherParams& p, cudaStream_t s, int num_sms);
}  // namespace kvev
