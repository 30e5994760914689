// api.cu -- host side of libkvev.so: the static plan (Sec. 3.1, Eq. 1), the
// capacity allocator (Sec. 3.3, Eq. 3), workspace layout, TMA descriptor
// encoding and the grouped launch sequence of the prefill eviction:
//   prologue (lengths, work items)  ->  window scores (tcgen05)  ->
//   selection (radix top-k)          ->  gather-compaction.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <memory>
#include <mutex>
#include <new>
#include <numeric>
#include <vector>

#include <cudaTypedefs.h>

#include "kvev_internal.cuh"

using namespace kvev;

// Per-device launch context: device properties, which kernel attributes were
// set, and the device status word the kernels report to.
struct DevCtx {
  int device = -1;
  int num_sms = 0;
  int smem_optin = 0;
  size_t score_smem_set = 0, h2o_full_smem_set = 0;
  int* status = nullptr;
};

struct kvev_plan {
  int L = 0, H_q = 0, H_kv = 0, d = 0, G = 0;
  int W = 0, pool_kernel = 1, pool_type = 0, sink = 0, recent = -1, h2o_recent = -1;
  std::vector<int> route_pre, route_dec, budget;
  std::vector<int> slots;       // output slots per (seq, head), 0 for FULL
  std::vector<int> recent_eff;  // StreamingLLM recent kept
  std::vector<int> h2o_r;       // H2O protected window
  std::vector<int> score_slot;  // index among scoring layers, -1 if none
  std::vector<int> score_layers;
  int64_t wait_ns = 2000000000LL;
  int stall_unit = -1;
  bool h2o_full = false;  // H2O prefill scores accumulate over every prompt query row
  // device-side state, created on first use (status word allocated lazily)
  DevCtx ctx;
  cudaStream_t last_stream = nullptr;
  // optional per-kernel timing of the last call
  bool timing = false;
  bool timed_call = false;
  cudaEvent_t ev[2 * KVEV_NUM_KERNELS] = {};
  bool launched[KVEV_NUM_KERNELS] = {};
};

namespace {

constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool is_scoring(int m) { return m == KVEV_SNAPKV || m == KVEV_H2O; }

struct WsLayout {
  int n_units = 0, R = 0, R_pad = 0, max_items = 0, n_h2o_units = 0;
  size_t lens = 0, abort_flag = 0, node_cnt = 0, ready = 0, chunk_start = 0, item = 0, part = 0,
         lam = 0, raw = 0, lse = 0, sel_keys = 0, total = 0;
};

// Entries of a selection key row: S_cap rounded up to whole 128-key blocks.
int sel_key_stride(int S_cap) { return (S_cap + 127) & ~127; }

WsLayout ws_layout(const kvev_plan& p, int B, int S_cap) {
  WsLayout w;
  w.n_units = static_cast<int>(p.score_layers.size()) * B * p.H_kv;
  w.R = p.G * p.W;
  w.R_pad = (w.R + 31) / 32 * 32;  // whole 32-column TMEM loads in the second sweep
  const int chunk_min = kTileKeys * kMinChunkTiles;
  w.max_items = w.n_units * ((S_cap + chunk_min - 1) / chunk_min);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, kWsAlign);
    return o;
  };
  w.lens = take(sizeof(int) * std::max(B, 1));
  w.abort_flag = take(sizeof(int));
  w.node_cnt = take(sizeof(int) * static_cast<size_t>(std::max(w.max_items, 1)) * kTreeLevels);
  w.ready = take(sizeof(int) * std::max(w.n_units, 1));
  w.chunk_start = take(sizeof(int) * (w.n_units + 1));
  w.item = take(sizeof(int4) * std::max(w.max_items, 1));
  w.part = take(sizeof(float2) * static_cast<size_t>(w.max_items) * w.R_pad);  // one per chunk
  w.lam = take(sizeof(float) * static_cast<size_t>(w.n_units) * w.R_pad);
  w.raw = take(sizeof(float) * static_cast<size_t>(w.n_units) * S_cap);
  // the selection's keys, one 16-byte aligned row per scoring unit
  w.sel_keys = take(sizeof(uint32_t) * static_cast<size_t>(w.n_units) * sel_key_stride(S_cap));
  if (p.h2o_full) {  // base-2 log-sum-exp of every prompt row of every H2O unit
    for (int l : p.score_layers) w.n_h2o_units += p.route_pre[l] == KVEV_H2O ? B * p.H_kv : 0;
    w.lse = take(sizeof(float) * static_cast<size_t>(w.n_h2o_units) * p.G * S_cap);
  }
  w.total = off;
  return w;
}

// Prompt positions per query block of the whole-prompt H2O kernels: as many
// as keep the block's G * Pb rows within two 128-lane row groups.
int prompt_block(int G) { return std::max(1, 256 / G); }

int64_t rows_per_layer(const kvev_plan& p, int B, int l) {
  return static_cast<int64_t>(B) * p.H_kv * p.slots[l];
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D bf16 map {d, rows} with a {64, box_rows} box and the 128-byte swizzle.
bool encode_map(CUtensorMap* m, const void* base, int d, uint64_t rows, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), rows};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Whole-prompt queries bf16 [B*H_q][S_cap][d] as a 3-D map whose box is G
// heads x W positions x 64 columns: it lands as the G*W rows of 128 bytes of
// a window (head-major), the layout of the 2-D window map.
bool encode_map_prompt(CUtensorMap* m, const void* base, int d, int S_cap, uint64_t heads, int W, int G) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(S_cap), heads};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(S_cap) * d * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(W), static_cast<cuuint32_t>(G)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Device properties of the current device into `c` (no allocation).
int query_device(DevCtx& c, int dev) {
  int major = 0;
  if (cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&c.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess)
    return KVEV_ECUDA;
  if (major < 10) return KVEV_ENOTSUP;
  c.device = dev;
  c.score_smem_set = c.h2o_full_smem_set = 0;
  return KVEV_OK;
}

int ensure_device(kvev_plan* p) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KVEV_ECUDA;
  DevCtx& c = p->ctx;
  if (c.device == dev && c.status) return KVEV_OK;
  if (c.status) {
    cudaFree(c.status);
    c.status = nullptr;
  }
  int rc = query_device(c, dev);
  if (rc != KVEV_OK) return rc;
  c.device = -1;
  if (cudaMalloc(&c.status, sizeof(int)) != cudaSuccess) return KVEV_ENOMEM;
  if (cudaMemset(c.status, 0, sizeof(int)) != cudaSuccess) return KVEV_ECUDA;
  c.device = dev;
  return KVEV_OK;
}

// Largest-remainder rounding of x (non-negative, sum == total): floor, then one
// extra unit to each of the largest fractional parts, lower index first on ties.
void round_largest_remainder(const std::vector<double>& x, int64_t total, int32_t* out) {
  const int L = static_cast<int>(x.size());
  std::vector<double> frac(L);
  int64_t sum = 0;
  for (int l = 0; l < L; ++l) {
    const double f = std::floor(x[l]);
    out[l] = static_cast<int32_t>(f);
    frac[l] = x[l] - f;
    sum += out[l];
  }
  std::vector<int> order(L);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(),
                   [&](int a, int b) { return frac[a] > frac[b]; });
  int64_t left = total - sum;
  for (int i = 0; i < L && left > 0; ++i, --left) out[order[i]] += 1;
}

}  // namespace

// ---------------------------------------------------------------------------
// Allocation (Sec. 3.3)
// ---------------------------------------------------------------------------

extern "C" int kvev_alloc_from_scores(int32_t* budget_out, const double* s, int L,
                                      int64_t B_total, int b_min, int transform) {
  if (!budget_out || !s || L <= 0 || b_min < 0 || static_cast<int64_t>(L) * b_min > B_total)
    return KVEV_EINVAL;
  if (transform != KVEV_T_IDENTITY && transform != KVEV_T_CAP_Q95) return KVEV_EINVAL;
  for (int l = 0; l < L; ++l)
    if (!std::isfinite(s[l])) return KVEV_EINVAL;
  std::vector<double> t(s, s + L);
  if (transform == KVEV_T_CAP_Q95) {
    std::vector<double> sorted(t);
    std::sort(sorted.begin(), sorted.end());
    const double h = 0.95 * (L - 1);
    const int lo = static_cast<int>(std::floor(h));
    double q = sorted[lo];
    if (lo + 1 < L) q += (h - lo) * (sorted[lo + 1] - sorted[lo]);
    for (double& v : t) v = std::min(v, q);
  }
  const double mn = *std::min_element(t.begin(), t.end());
  if (mn <= 0.0)
    for (double& v : t) v += -mn + 1e-6;
  double tsum = 0.0;
  for (double v : t) tsum += v;
  std::vector<double> w(L), bt(L);
  for (int l = 0; l < L; ++l) w[l] = t[l] / tsum;
  std::vector<char> fixed(L, 0);
  bool changed = true;
  while (changed) {
    changed = false;
    int nfixed = 0;
    double wfree = 0.0;
    for (int l = 0; l < L; ++l) {
      if (fixed[l]) ++nfixed;
      else wfree += w[l];
    }
    const double rest = static_cast<double>(B_total) - static_cast<double>(nfixed) * b_min;
    for (int l = 0; l < L; ++l)
      bt[l] = fixed[l] ? static_cast<double>(b_min) : (wfree > 0.0 ? rest * w[l] / wfree : 0.0);
    for (int l = 0; l < L; ++l)
      if (!fixed[l] && bt[l] < static_cast<double>(b_min)) fixed[l] = 1, changed = true;
  }
  round_largest_remainder(bt, B_total, budget_out);
  return KVEV_OK;
}

extern "C" int kvev_alloc_rescale(int32_t* budget_out, const int32_t* budget_in, int L,
                                  int64_t B_target) {
  if (!budget_out || !budget_in || L <= 0 || B_target < 0) return KVEV_EINVAL;
  int64_t sum = 0;
  for (int l = 0; l < L; ++l) {
    if (budget_in[l] < 0) return KVEV_EINVAL;
    sum += budget_in[l];
  }
  if (sum <= 0) return KVEV_EINVAL;
  std::vector<double> x(L);
  for (int l = 0; l < L; ++l)
    x[l] = static_cast<double>(budget_in[l]) * (static_cast<double>(B_target) / sum);
  round_largest_remainder(x, B_target, budget_out);
  return KVEV_OK;
}

// ---------------------------------------------------------------------------
// Plan
// ---------------------------------------------------------------------------

extern "C" int kvev_plan_create(kvev_plan** out, int L, int H_q, int H_kv, int d,
                                const int32_t* route_prefill, const int32_t* route_decode,
                                const int32_t* budget, int window, int pool_kernel,
                                int pool_type, int sink, int recent, int h2o_recent) {
  if (!out) return KVEV_EINVAL;
  *out = nullptr;
  if (L <= 0 || H_q <= 0 || H_kv <= 0 || H_q % H_kv != 0 || d <= 0 || !route_prefill || !budget)
    return KVEV_EINVAL;
  if (L > kMaxLayers) return KVEV_ENOTSUP;
  if (pool_type != KVEV_POOL_MAX && pool_type != KVEV_POOL_AVG) return KVEV_EINVAL;
  std::unique_ptr<kvev_plan> p(new (std::nothrow) kvev_plan);
  if (!p) return KVEV_ENOMEM;
  p->L = L;
  p->H_q = H_q;
  p->H_kv = H_kv;
  p->d = d;
  p->G = H_q / H_kv;
  p->W = window;
  p->pool_kernel = pool_kernel;
  p->pool_type = pool_type;
  p->sink = sink;
  p->recent = recent;
  p->h2o_recent = h2o_recent;
  p->route_pre.assign(route_prefill, route_prefill + L);
  p->budget.assign(budget, budget + L);
  p->route_dec.assign(L, KVEV_FULL);
  if (route_decode) p->route_dec.assign(route_decode, route_decode + L);
  p->slots.assign(L, 0);
  p->recent_eff.assign(L, 0);
  p->h2o_r.assign(L, 0);
  p->score_slot.assign(L, -1);
  bool any_scoring = false, any_snap = false;
  for (int l = 0; l < L; ++l) {
    const int m = p->route_pre[l], b = p->budget[l];
    switch (m) {
      case KVEV_FULL:
        break;
      case KVEV_SNAPKV:
        if (b <= window) return KVEV_EINVAL;
        any_snap = any_scoring = true;
        break;
      case KVEV_H2O: {
        const int r = h2o_recent < 0 ? b / 2 : h2o_recent;
        if (b < 1 || r > b) return KVEV_EINVAL;
        p->h2o_r[l] = r;
        any_scoring = true;
        break;
      }
      case KVEV_STREAMING:
        if (sink < 0 || b <= sink) return KVEV_EINVAL;
        p->recent_eff[l] = recent < 0 ? b - sink : std::min(recent, b - sink);
        break;
      default:
        return KVEV_EINVAL;
    }
    if (m != KVEV_FULL) p->slots[l] = b;
    if (is_scoring(m)) {
      p->score_slot[l] = static_cast<int>(p->score_layers.size());
      p->score_layers.push_back(l);
    }
    const int md = p->route_dec[l];
    if (md != KVEV_FULL && md != KVEV_H2O && md != KVEV_TOVA && md != KVEV_STREAMING)
      return KVEV_EINVAL;
  }
  if (any_snap && (pool_kernel < 1 || (pool_kernel & 1) == 0)) return KVEV_EINVAL;
  if (any_scoring) {
    if (window < 1) return KVEV_EINVAL;
    if (d != 64 && d != 128) return KVEV_ENOTSUP;
    if (p->G * window > 256) return KVEV_ENOTSUP;
    if (static_cast<int>(p->score_layers.size()) > kMaxScoreLayers) return KVEV_ENOTSUP;
  }
  if (d % 8 != 0) return KVEV_ENOTSUP;  // 16-byte row vectors in the gather
  *out = p.release();
  return KVEV_OK;
}

// ---- plan serialisation (Sec. 3.4) ------------------------------------------
namespace {

constexpr char kPlanMagic[8] = {'K', 'V', 'E', 'V', 'P', 'L', 'N', '1'};
constexpr int kPlanHead = 10;  // words after the magic: L, H_q, H_kv, d, W, pool, type, sink, recent, h2o

uint64_t fnv1a(const uint8_t* p, size_t n) {
  uint64_t h = 1469598103934665603ULL;
  for (size_t i = 0; i < n; ++i) {
    h ^= p[i];
    h *= 1099511628211ULL;
  }
  return h;
}

size_t plan_bytes(int L) { return 8 + 4 * static_cast<size_t>(kPlanHead + 3 * L) + 8; }

void put32(uint8_t* p, uint32_t v) {
  for (int i = 0; i < 4; ++i) p[i] = static_cast<uint8_t>(v >> (8 * i));
}
uint32_t get32(const uint8_t* p) {
  uint32_t v = 0;
  for (int i = 0; i < 4; ++i) v |= static_cast<uint32_t>(p[i]) << (8 * i);
  return v;
}

}  // namespace

extern "C" int kvev_plan_save(const kvev_plan* plan, void* buf, size_t* bytes) {
  if (!plan || !bytes) return KVEV_EINVAL;
  const kvev_plan& P = *plan;
  const size_t need = plan_bytes(P.L);
  if (!buf) {
    *bytes = need;
    return KVEV_OK;
  }
  if (*bytes < need) return KVEV_EINVAL;
  uint8_t* o = static_cast<uint8_t*>(buf);
  std::memcpy(o, kPlanMagic, 8);
  size_t at = 8;
  const int32_t head[kPlanHead] = {P.L, P.H_q, P.H_kv, P.d, P.W, P.pool_kernel, P.pool_type,
                                   P.sink, P.recent, P.h2o_recent};
  for (int i = 0; i < kPlanHead; ++i, at += 4) put32(o + at, static_cast<uint32_t>(head[i]));
  for (const std::vector<int>* v : {&P.route_pre, &P.route_dec, &P.budget})
    for (int l = 0; l < P.L; ++l, at += 4) put32(o + at, static_cast<uint32_t>((*v)[l]));
  const uint64_t h = fnv1a(o, at);
  put32(o + at, static_cast<uint32_t>(h));
  put32(o + at + 4, static_cast<uint32_t>(h >> 32));
  *bytes = need;
  return KVEV_OK;
}

extern "C" int kvev_plan_load(kvev_plan** out, const void* buf, size_t bytes) {
  if (!out) return KVEV_EINVAL;
  *out = nullptr;
  if (!buf || bytes < 8 + 4 * kPlanHead + 8) return KVEV_EINVAL;
  const uint8_t* in = static_cast<const uint8_t*>(buf);
  if (std::memcmp(in, kPlanMagic, 8) != 0) return KVEV_EINVAL;
  const int32_t L = static_cast<int32_t>(get32(in + 8));
  if (L <= 0 || L > kMaxLayers || bytes != plan_bytes(L)) return KVEV_EINVAL;
  const size_t body = bytes - 8;
  const uint64_t h = static_cast<uint64_t>(get32(in + body)) | (static_cast<uint64_t>(get32(in + body + 4)) << 32);
  if (h != fnv1a(in, body)) return KVEV_EINVAL;
  int32_t head[kPlanHead];
  for (int i = 0; i < kPlanHead; ++i) head[i] = static_cast<int32_t>(get32(in + 8 + 4 * i));
  std::vector<int32_t> pre(L), dec(L), bud(L);
  size_t at = 8 + 4 * kPlanHead;
  for (std::vector<int32_t>* v : {&pre, &dec, &bud})
    for (int l = 0; l < L; ++l, at += 4) (*v)[l] = static_cast<int32_t>(get32(in + at));
  return kvev_plan_create(out, L, head[1], head[2], head[3], pre.data(), dec.data(), bud.data(), head[4],
                          head[5], head[6], head[7], head[8], head[9]);
}

extern "C" void kvev_plan_destroy(kvev_plan* plan) {
  if (!plan) return;
  if (plan->ctx.status) cudaFree(plan->ctx.status);
  for (cudaEvent_t e : plan->ev)
    if (e) cudaEventDestroy(e);
  delete plan;
}

extern "C" int kvev_plan_enable_timing(kvev_plan* plan, int on) {
  if (!plan) return KVEV_EINVAL;
  if (on && !plan->ev[0]) {
    for (cudaEvent_t& e : plan->ev)
      if (cudaEventCreate(&e) != cudaSuccess) return KVEV_ECUDA;
  }
  plan->timing = on != 0;
  plan->timed_call = false;
  return KVEV_OK;
}

extern "C" int kvev_plan_last_timings(kvev_plan* plan, float* ms, int n) {
  if (!plan || !ms || n < 0 || !plan->timing || !plan->timed_call) return KVEV_EINVAL;
  int last = -1;
  for (int k = 0; k < KVEV_NUM_KERNELS; ++k)
    if (plan->launched[k]) last = k;
  if (last >= 0 && cudaEventSynchronize(plan->ev[2 * last + 1]) != cudaSuccess) return KVEV_ECUDA;
  for (int k = 0; k < n && k < KVEV_NUM_KERNELS; ++k) {
    ms[k] = -1.f;
    if (plan->launched[k] &&
        cudaEventElapsedTime(&ms[k], plan->ev[2 * k], plan->ev[2 * k + 1]) != cudaSuccess)
      return KVEV_ECUDA;
  }
  return KVEV_OK;
}

extern "C" int kvev_plan_query(const kvev_plan* plan, int B, int S_cap, size_t* out_kv_bytes,
                               size_t* out_idx_bytes, size_t* count_bytes,
                               size_t* workspace_bytes) {
  if (!plan || B < 0 || S_cap < 1) return KVEV_EINVAL;
  int64_t rows = 0;
  for (int l = 0; l < plan->L; ++l) rows += rows_per_layer(*plan, B, l);
  if (out_kv_bytes) *out_kv_bytes = static_cast<size_t>(rows) * plan->d * 2;
  if (out_idx_bytes) *out_idx_bytes = static_cast<size_t>(rows) * sizeof(int32_t);
  if (count_bytes) *count_bytes = static_cast<size_t>(plan->L) * B * plan->H_kv * sizeof(int32_t);
  if (workspace_bytes) *workspace_bytes = ws_layout(*plan, B, S_cap).total;
  return KVEV_OK;
}

extern "C" int kvev_plan_layer_offset(const kvev_plan* plan, int B, int layer,
                                      int64_t* row_offset) {
  if (!plan || !row_offset || B < 0 || layer < 0 || layer >= plan->L) return KVEV_EINVAL;
  int64_t off = 0;
  for (int l = 0; l < layer; ++l) off += rows_per_layer(*plan, B, l);
  *row_offset = off;
  return KVEV_OK;
}

extern "C" int kvev_plan_scores_offset(const kvev_plan* plan, int B, int S_cap, int layer,
                                       size_t* byte_offset) {
  if (!plan || !byte_offset || B < 0 || S_cap < 1 || layer < 0 || layer >= plan->L ||
      plan->score_slot[layer] < 0)
    return KVEV_EINVAL;
  const WsLayout ws = ws_layout(*plan, B, S_cap);
  *byte_offset = ws.raw + sizeof(float) * static_cast<size_t>(plan->score_slot[layer]) * B *
                              plan->H_kv * S_cap;
  return KVEV_OK;
}

extern "C" int kvev_plan_set_h2o_full_prompt(kvev_plan* plan, int on) {
  if (!plan || (on != 0 && on != 1)) return KVEV_EINVAL;
  plan->h2o_full = on == 1;
  return KVEV_OK;
}

extern "C" int kvev_plan_set_wait_limit(kvev_plan* plan, int64_t ns) {
  if (!plan || ns <= 0) return KVEV_EINVAL;
  plan->wait_ns = ns;
  return KVEV_OK;
}

extern "C" int kvev_plan_debug_stall_unit(kvev_plan* plan, int unit) {
  if (!plan) return KVEV_EINVAL;
  plan->stall_unit = unit;
  return KVEV_OK;
}

extern "C" int kvev_status(kvev_plan* plan, int* device_status) {
  if (!plan || !device_status) return KVEV_EINVAL;
  *device_status = KVEV_OK;
  if (!plan->ctx.status) return KVEV_OK;
  if (cudaStreamSynchronize(plan->last_stream) != cudaSuccess) return KVEV_ECUDA;
  int v = 0;
  if (cudaMemcpy(&v, plan->ctx.status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemset(plan->ctx.status, 0, sizeof(int)) != cudaSuccess)
    return KVEV_ECUDA;
  *device_status = (v & kStatusTimeout) ? KVEV_ETIMEOUT : (v & kStatusDevice) ? KVEV_EDEVICE : 0;
  return KVEV_OK;
}

// ---------------------------------------------------------------------------
// Prefill eviction
// ---------------------------------------------------------------------------

namespace {

// Argument checks shared by the prefill entry points (no device work).
int check_prefill_args(const kvev_plan& P, const void* const* K, const void* const* V,
                       const void* const* Q_win, const float* const* scores, const int32_t* lens_dev,
                       int B, int S_cap, void* out_K, void* out_V, int32_t* out_idx,
                       int32_t* out_count) {
  if (!K || !V || !lens_dev || !out_count) return KVEV_EINVAL;
  if (static_cast<int64_t>(B) * P.H_kv * S_cap > (1LL << 31) - 1) return KVEV_ENOTSUP;
  int64_t total_rows = 0;
  for (int l = 0; l < P.L; ++l) total_rows += rows_per_layer(P, B, l);
  if (total_rows > 0 && (!out_K || !out_V || !out_idx)) return KVEV_EINVAL;
  if (!aligned16(out_K) || !aligned16(out_V)) return KVEV_EINVAL;
  for (int l = 0; l < P.L; ++l) {
    if (P.route_pre[l] == KVEV_FULL) continue;
    if (!K[l] || !V[l] || !aligned16(K[l]) || !aligned16(V[l])) return KVEV_EINVAL;
    if (!is_scoring(P.route_pre[l])) continue;
    if (scores && scores[l]) {  // supplied by the caller: Q_win[l] is not read
      if (reinterpret_cast<uintptr_t>(scores[l]) & 3u) return KVEV_EINVAL;
    } else if (!Q_win || !Q_win[l] || !aligned16(Q_win[l])) {
      return KVEV_EINVAL;
    }
  }
  return KVEV_OK;
}

// The launch sequence of one prefill eviction, given a validated argument set,
// a device context (properties + status word) and a scratch workspace of at
// least ws_layout(P, B, S_cap).total bytes (256-byte aligned).
int evict_impl(kvev_plan& P, DevCtx& D, const void* const* K, const void* const* V,
               const void* const* Q_win, const float* const* scores, const int32_t* lens_dev, int B,
               int S_cap, void* out_K, void* out_V, int32_t* out_idx, int32_t* out_count,
               float* h2o_state, void* workspace, cudaStream_t s, const float* const* lse_win = nullptr);

int evict_prefill_impl(kvev_plan* plan, const void* const* K, const void* const* V,
                       const void* const* Q_win, const float* const* scores, const int32_t* lens_dev,
                       int B, int S_cap, void* out_K, void* out_V, int32_t* out_idx,
                       int32_t* out_count, float* h2o_state, void* workspace, size_t workspace_bytes,
                       void* stream, const float* const* lse_win = nullptr) {
  if (!plan || B < 0 || S_cap < 1) return KVEV_EINVAL;
  kvev_plan& P = *plan;
  if (B == 0) return KVEV_OK;
  int rc = check_prefill_args(P, K, V, Q_win, scores, lens_dev, B, S_cap, out_K, out_V, out_idx,
                              out_count);
  if (rc != KVEV_OK) return rc;
  if (lse_win) {  // every scored layer needs its rows' log-sum-exp
    for (int l = 0; l < P.L; ++l)
      if (is_scoring(P.route_pre[l]) &&
          (!lse_win[l] || (reinterpret_cast<uintptr_t>(lse_win[l]) & 3u)))
        return KVEV_EINVAL;
  }
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return KVEV_EINVAL;
  if (workspace_bytes < ws_layout(P, B, S_cap).total) return KVEV_ENOMEM;
  rc = ensure_device(plan);
  if (rc != KVEV_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  P.last_stream = s;
  return evict_impl(P, P.ctx, K, V, Q_win, scores, lens_dev, B, S_cap, out_K, out_V, out_idx,
                    out_count, h2o_state, workspace, s, lse_win);
}

}  // namespace

extern "C" int kvev_evict_prefill(kvev_plan* plan, const void* const* K, const void* const* V,
                                  const void* const* Q_win, const int32_t* lens_dev, int B,
                                  int S_cap, void* out_K, void* out_V, int32_t* out_idx,
                                  int32_t* out_count, float* h2o_state, void* workspace,
                                  size_t workspace_bytes, void* stream) {
  return evict_prefill_impl(plan, K, V, Q_win, nullptr, lens_dev, B, S_cap, out_K, out_V, out_idx,
                            out_count, h2o_state, workspace, workspace_bytes, stream);
}

extern "C" int kvev_evict_prefill_scored(kvev_plan* plan, const void* const* K, const void* const* V,
                                         const void* const* Q_win, const float* const* scores,
                                         const int32_t* lens_dev, int B, int S_cap, void* out_K,
                                         void* out_V, int32_t* out_idx, int32_t* out_count,
                                         float* h2o_state, void* workspace, size_t workspace_bytes,
                                         void* stream) {
  if (!scores) return KVEV_EINVAL;
  return evict_prefill_impl(plan, K, V, Q_win, scores, lens_dev, B, S_cap, out_K, out_V, out_idx,
                            out_count, h2o_state, workspace, workspace_bytes, stream);
}

extern "C" int kvev_evict_prefill_lse(kvev_plan* plan, const void* const* K, const void* const* V,
                                      const void* const* Q_win, const float* const* lse_win,
                                      const int32_t* lens_dev, int B, int S_cap, void* out_K,
                                      void* out_V, int32_t* out_idx, int32_t* out_count,
                                      float* h2o_state, void* workspace, size_t workspace_bytes,
                                      void* stream) {
  if (!lse_win) return KVEV_EINVAL;
  return evict_prefill_impl(plan, K, V, Q_win, nullptr, lens_dev, B, S_cap, out_K, out_V, out_idx,
                            out_count, h2o_state, workspace, workspace_bytes, stream, lse_win);
}

namespace {

// 1 when the compiled score kernel for head size d is launched with enough
// registers for its setmaxnreg split, 0 when not, -1 when the query failed.
int score_regs_ok(int d) {
  static std::once_flag once[2];
  static int ok[2] = {-1, -1};
  const int i = d == 64 ? 0 : 1;
  std::call_once(once[i], [&] {
    const int regs = score_kernel_regs(d);
    ok[i] = regs < 0 ? -1 : (regs * kScoreThreads >= kRegsNeeded ? 1 : 0);
  });
  return ok[i];
}

// The same check for the whole-prompt H2O kernel (same warp roles and split).
int h2o_full_regs_ok(int d) {
  static std::once_flag once[2];
  static int ok[2] = {-1, -1};
  const int i = d == 64 ? 0 : 1;
  std::call_once(once[i], [&] {
    const int regs = h2o_full_kernel_regs(d);
    ok[i] = regs < 0 ? -1 : (regs * kScoreThreads >= kRegsNeeded ? 1 : 0);
  });
  return ok[i];
}

int evict_impl(kvev_plan& P, DevCtx& D, const void* const* K, const void* const* V,
               const void* const* Q_win, const float* const* scores, const int32_t* lens_dev, int B,
               int S_cap, void* out_K, void* out_V, int32_t* out_idx, int32_t* out_count,
               float* h2o_state, void* workspace, cudaStream_t s, const float* const* lse_win) {
  auto supplied = [&](int l) { return scores != nullptr && scores[l] != nullptr; };
  if (static_cast<int64_t>(B) * P.H_kv * S_cap > (1LL << 31) - 1) return KVEV_ENOTSUP;
  const WsLayout ws = ws_layout(P, B, S_cap);
  uint8_t* wsb = static_cast<uint8_t*>(workspace);
  int* lens_ok = reinterpret_cast<int*>(wsb + ws.lens);

  // ---- prologue: validated lengths, work items, flag reset -------------
  const int n_slayers = static_cast<int>(P.score_layers.size());
  // chunk size: at least kMinChunkTiles tiles, and few enough chunks per unit
  // that a unit never spans more than two rounds of the persistent grid
  const int grid = D.num_sms;
  const int tiles_max = (S_cap + kTileKeys - 1) / kTileKeys;
  // (an even number of tiles: chunks are swept in 256-key super-tiles)
  const int chunk_tiles = (std::max(kMinChunkTiles, (tiles_max + grid - 1) / grid) + 1) & ~1;
  if (chunk_tiles > 0xFFFF) return KVEV_ENOTSUP;  // tiles per item are packed in 16 bits
  // the normaliser's merge tree has kTreeLevels internal levels of fan-in kTreeFanIn
  int leaves = 1;
  for (int i = 0; i < kTreeLevels; ++i) leaves *= kTreeFanIn;
  if ((tiles_max + chunk_tiles - 1) / chunk_tiles > leaves) return KVEV_ENOTSUP;
  PrologueParams pp = {};
  pp.n_units = ws.n_units;
  pp.B = B;
  pp.H_kv = P.H_kv;
  pp.chunk_keys = chunk_tiles * kTileKeys;
  for (int i = 0; i < n_slayers; ++i) {
    pp.slayer_method[i] = P.route_pre[P.score_layers[i]];
    pp.slayer_budget[i] = P.budget[P.score_layers[i]];
    pp.slayer_ext[i] = supplied(P.score_layers[i]) ? 1 : 0;
  }
  pp.lens_in = lens_dev;
  pp.lens = lens_ok;
  pp.S_cap = S_cap;
  pp.status = D.status;
  pp.node_cnt = reinterpret_cast<int*>(wsb + ws.node_cnt);
  pp.n_node_cnt = std::max(ws.max_items, 1) * kTreeLevels;
  pp.ready = reinterpret_cast<int*>(wsb + ws.ready);
  pp.abort_flag = reinterpret_cast<int*>(wsb + ws.abort_flag);
  pp.chunk_start = reinterpret_cast<int*>(wsb + ws.chunk_start);
  pp.item = reinterpret_cast<int4*>(wsb + ws.item);
  for (bool& b : P.launched) b = false;
  P.timed_call = P.timing;
  auto mark = [&](int k, int which) {
    if (P.timing) {
      cudaEventRecord(P.ev[2 * k + which], s);
      if (which == 1) P.launched[k] = true;
    }
  };
  pp.W = P.W;
  bool any_h2o = false;
  for (int i = 0; i < n_slayers; ++i)
    any_h2o |= P.route_pre[P.score_layers[i]] == KVEV_H2O && !supplied(P.score_layers[i]);
  // H2O prefill scores over every prompt query row: the window kernel scores
  // the SnapKV layers only, and the whole-prompt kernels the H2O layers
  const bool full_prompt = P.h2o_full && any_h2o;

  // ---- window scores ----------------------------------------------------
  ScoreParams sp;
  std::memset(&sp, 0, sizeof(sp));
  int score_grid = 0;
  size_t score_smem = 0;
  if (ws.n_units > 0) {
    const int q_rows = ws.R_pad > 128 ? 256 : 128;
    for (int i = 0; i < n_slayers; ++i) {
      const int l = P.score_layers[i];
      if (supplied(l)) continue;  // not scored here: its maps are never used
      if (!encode_map(&sp.kmap[i], K[l], P.d, static_cast<uint64_t>(B) * P.H_kv * S_cap,
                      kSuperKeys) ||
          !(full_prompt && P.route_pre[l] == KVEV_H2O
                ? encode_map_prompt(&sp.qmap[i], Q_win[l], P.d, S_cap, static_cast<uint64_t>(B) * P.H_q,
                                    prompt_block(P.G), P.G)
                : encode_map(&sp.qmap[i], Q_win[l], P.d, static_cast<uint64_t>(B) * P.H_q * P.W,
                             ws.R_pad)))
        return KVEV_ECUDA;
    }
    // K stages (256-key super-tiles) that fit next to q_bufs Q buffers.  A
    // second Q buffer hides the next entry's Q load, but the ring needs two
    // stages; with one buffer the next entry's Q loads once this one is done.
    auto fit = [&](int q_bufs) {
      int st = 4;
      while (st >= 2 && score_smem_bytes(P.d, q_rows, q_bufs, ws.R_pad, st) + 1024 > D.smem_optin)
        --st;
      return st;
    };
    int q_bufs = 2, stages = fit(2);
    if (stages < 2) {
      q_bufs = 1;
      stages = fit(1);
    }
    if (stages < 2) return KVEV_ENOTSUP;
    // The softmax warpgroups raise their register count with setmaxnreg,
    // drawing on the registers the CTA was launched with; refuse to launch a
    // build whose allocation could not cover that (the raise would never
    // complete).
    if (score_regs_ok(P.d) != 1) return KVEV_ENOTSUP;
    // Request more than half of the SM's shared memory so exactly one CTA is
    // resident per SM: its TMEM allocation then never waits on another CTA.
    const size_t smem = std::max<size_t>(score_smem_bytes(P.d, q_rows, q_bufs, ws.R_pad, stages),
                                         static_cast<size_t>(D.smem_optin) / 2 + 1024);
    if (D.score_smem_set != smem) {
      if (score_set_smem(P.d, smem) != cudaSuccess) return KVEV_ECUDA;
      D.score_smem_set = smem;
    }
    sp.n_units = ws.n_units;
    sp.B = B;
    sp.H_kv = P.H_kv;
    sp.H_q = P.H_q;
    sp.G = P.G;
    sp.W = P.W;
    sp.R = ws.R;
    sp.R_pad = ws.R_pad;
    sp.S_cap = S_cap;
    sp.chunk_keys = pp.chunk_keys;
    sp.q_rows = q_rows;
    sp.q_bufs = q_bufs;
    sp.stages = stages;
    sp.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(P.d)));
    sp.inv_G = 1.0f / static_cast<float>(P.G);
    sp.lens = lens_ok;
    sp.chunk_start = pp.chunk_start;
    sp.item = pp.item;
    sp.node_cnt = pp.node_cnt;
    sp.ready = pp.ready;
    sp.abort_flag = pp.abort_flag;
    sp.status = D.status;
    sp.part = reinterpret_cast<float2*>(wsb + ws.part);
    sp.lam = reinterpret_cast<float*>(wsb + ws.lam);
    sp.raw = reinterpret_cast<float*>(wsb + ws.raw);
    sp.wait_ns = P.wait_ns;
    sp.stall_unit = P.stall_unit;
    sp.single = lse_win ? 1 : 0;
    score_grid = grid;
    score_smem = smem;
  }
  mark(KVEV_K_PROLOGUE, 0);
  pp.mode = full_prompt ? kScoreNoH2O : kScoreAll;
  if (launch_prologue(pp, s) != cudaSuccess) return KVEV_ECUDA;
  if (lse_win && ws.n_units > 0) {  // the caller's normalisers: the score kernel makes one sweep
    LseParams lp;
    std::memset(&lp, 0, sizeof(lp));
    for (int i = 0; i < n_slayers; ++i) {  // H2O layers scored over the whole prompt: below
      const int l = P.score_layers[i];
      lp.lse[i] = supplied(l) || (full_prompt && P.route_pre[l] == KVEV_H2O) ? nullptr : lse_win[l];
    }
    lp.n_units = ws.n_units;
    lp.B = B;
    lp.H_kv = P.H_kv;
    lp.H_q = P.H_q;
    lp.G = P.G;
    lp.W = P.W;
    lp.R = ws.R;
    lp.R_pad = ws.R_pad;
    lp.lens = lens_ok;
    lp.lam = reinterpret_cast<float*>(wsb + ws.lam);
    lp.ready = reinterpret_cast<int*>(wsb + ws.ready);
    if (launch_lse_fill(lp, s) != cudaSuccess) return KVEV_ECUDA;
  }
  mark(KVEV_K_PROLOGUE, 1);
  if (ws.n_units > 0) mark(KVEV_K_SCORE, 0);
  if (ws.n_units > 0 &&
      launch_score(sp, P.d, score_grid, score_smem, s) != cudaSuccess)
    return KVEV_ECUDA;
  if (full_prompt) {
    // row pass (lse2 of every prompt row), then key pass (the scores)
    ScoreParams fp = sp;
    fp.Pb = prompt_block(P.G);
    fp.R = P.G * fp.Pb;
    fp.R_pad = (fp.R + 31) / 32 * 32;
    fp.n_h2o = 0;
    for (int i = 0; i < n_slayers; ++i)
      if (P.route_pre[P.score_layers[i]] == KVEV_H2O && !supplied(P.score_layers[i]))
        fp.h2o_slot[fp.n_h2o++] = i;
    fp.nb_max = (S_cap + fp.Pb - 1) / fp.Pb;
    fp.nkt_max = (S_cap + kSuperKeys - 1) / kSuperKeys;
    fp.lse = reinterpret_cast<float*>(wsb + ws.lse);
    const int64_t units = static_cast<int64_t>(fp.n_h2o) * B * P.H_kv;
    if (units * std::max(fp.nb_max, fp.nkt_max) > (1LL << 31) - 1) return KVEV_ENOTSUP;
    if (h2o_full_regs_ok(P.d) != 1) return KVEV_ENOTSUP;
    // more than half of the SM's shared memory: one CTA per SM, so its TMEM
    // allocation never waits on another CTA
    const size_t fsmem = std::max<size_t>(static_cast<size_t>(h2o_full_smem_bytes(P.d)),
                                          static_cast<size_t>(D.smem_optin) / 2 + 1024);
    if (fsmem + 1024 > static_cast<size_t>(D.smem_optin)) return KVEV_ENOTSUP;
    if (D.h2o_full_smem_set != fsmem) {
      if (h2o_full_set_smem(P.d, fsmem) != cudaSuccess) return KVEV_ECUDA;
      D.h2o_full_smem_set = fsmem;
    }
    if (lse_win) {  // the caller's every-row normalisers replace the row pass
      for (int j = 0; j < fp.n_h2o; ++j) fp.lse_src[j] = lse_win[P.score_layers[fp.h2o_slot[j]]];
      if (launch_lse_rows_fill(fp, s) != cudaSuccess) return KVEV_ECUDA;
    }
    for (int phase = lse_win ? 1 : 0; phase < 2; ++phase) {
      fp.phase = phase;
      fp.n_items = static_cast<int>(units * (phase == 0 ? fp.nb_max : fp.nkt_max));
      if (launch_h2o_full(fp, P.d, std::min(D.num_sms, fp.n_items), fsmem, s) != cudaSuccess)
        return KVEV_ECUDA;
    }
  }
  if (ws.n_units > 0) mark(KVEV_K_SCORE, 1);

  // ---- selection --------------------------------------------------------
  SelectParams sel;
  std::memset(&sel, 0, sizeof(sel));
  GatherParams ga;
  std::memset(&ga, 0, sizeof(ga));
  int64_t off = 0, goff = 0;
  for (int l = 0; l < P.L; ++l) {
    LayerDesc ld;
    ld.method = P.route_pre[l];
    ld.slots = P.slots[l];
    ld.recent = P.recent_eff[l];
    ld.h2o_recent = P.h2o_r[l];
    ld.score_slot = P.score_slot[l];
    ld.row_off = off;
    ld.scores = nullptr;
    if (ld.score_slot >= 0)
      ld.scores = supplied(l) ? scores[l]
                              : reinterpret_cast<const float*>(wsb + ws.raw) +
                                    static_cast<size_t>(ld.score_slot) * B * P.H_kv * S_cap;
    ga.grow_off[l] = goff;
    if (is_scoring(ld.method)) goff += rows_per_layer(P, B, l);  // StreamingLLM rows: selection launch
    off += rows_per_layer(P, B, l);
    sel.layer[l] = ld;
    ga.layer[l] = ld;
    ga.K[l] = sel.K[l] = K[l];
    ga.V[l] = sel.V[l] = V[l];
  }
  for (int l = 0; l < P.L; ++l)  // selection dispatch: scoring layers first
    if (is_scoring(P.route_pre[l])) sel.order[sel.L_first++] = l;
  for (int l = 0, j = sel.L_first; l < P.L; ++l)
    if (!is_scoring(P.route_pre[l])) sel.order[j++] = l;
  sel.L = P.L;
  sel.B = B;
  sel.H_kv = P.H_kv;
  sel.S_cap = S_cap;
  sel.W = P.W;
  sel.pool_kernel = P.pool_kernel;
  sel.pool_type = P.pool_type;
  sel.sink = P.sink;
  sel.d = P.d;
  sel.out_K = out_K;
  sel.out_V = out_V;
  sel.lens = lens_ok;
  sel.out_idx = out_idx;
  sel.out_count = out_count;
  sel.keys = reinterpret_cast<uint32_t*>(wsb + ws.sel_keys);
  sel.key_stride = sel_key_stride(S_cap);
  mark(KVEV_K_SELECT, 0);
  if (launch_select(sel, P.L * B * P.H_kv, s) != cudaSuccess) return KVEV_ECUDA;
  mark(KVEV_K_SELECT, 1);

  // ---- gather-compaction ---------------------------------------------------
  ga.L = P.L;
  ga.B = B;
  ga.H_kv = P.H_kv;
  ga.S_cap = S_cap;
  ga.d = P.d;
  ga.total_rows = goff;
  ga.out_idx = out_idx;
  ga.out_K = out_K;
  ga.out_V = out_V;
  ga.h2o_state = h2o_state;
  ga.status = D.status;
  mark(KVEV_K_GATHER, 0);
  if (launch_gather(ga, s, D.num_sms) != cudaSuccess) return KVEV_ECUDA;
  if (goff > 0) mark(KVEV_K_GATHER, 1);
  return KVEV_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// Decode phase
// ---------------------------------------------------------------------------

namespace {

struct DecLayout {
  int units = 0;
  int64_t rows = 0;
  size_t lens = 0, count = 0, evicted = 0, pos = 0, acc = 0, done = 0, total = 0;
  std::vector<int> cap, unit_off;
  std::vector<int64_t> row_off;
};

// Arena layout for B sequences; growth = extra slots of append-only layers.
// Returns KVEV_EINVAL for a layer that has a decode-phase rule but no
// retained rows (a FULL prefill layer keeps the caller's own cache).
int dec_layout(const kvev_plan& P, int B, int growth, DecLayout& d) {
  if (B < 0 || growth < 0) return KVEV_EINVAL;
  d.cap.assign(P.L, 0);
  d.unit_off.assign(P.L, 0);
  d.row_off.assign(P.L, 0);
  for (int l = 0; l < P.L; ++l) {
    const int md = P.route_dec[l];
    d.unit_off[l] = d.units;
    d.row_off[l] = d.rows;
    if (P.slots[l] == 0) {
      if (md != KVEV_FULL) return KVEV_EINVAL;
      continue;
    }
    d.cap[l] = P.slots[l] + (md == KVEV_FULL ? growth : 0);
    d.units += B * P.H_kv;
    d.rows += static_cast<int64_t>(B) * P.H_kv * d.cap[l];
  }
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, kWsAlign);
    return o;
  };
  d.lens = take(sizeof(int32_t) * std::max(B, 1));
  d.count = take(sizeof(int32_t) * std::max(d.units, 1));
  d.evicted = take(sizeof(int32_t) * std::max(d.units, 1));
  d.pos = take(sizeof(int32_t) * std::max<int64_t>(d.rows, 1));
  d.acc = take(sizeof(float) * std::max<int64_t>(d.rows, 1));
  d.done = take(sizeof(int32_t));  // units finished in the current step (internal)
  d.total = off;
  return KVEV_OK;
}

int dec_params(const kvev_plan& P, int B, const DecLayout& d, DecodeParams& dp) {
  std::memset(&dp, 0, sizeof(dp));
  dp.L = P.L;
  dp.B = B;
  dp.H_kv = P.H_kv;
  dp.H_q = P.H_q;
  dp.G = P.G;
  dp.d = P.d;
  dp.units = d.units;
  dp.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(P.d)));
  int64_t pre_off = 0;
  for (int l = 0; l < P.L; ++l) {
    DecLayer& y = dp.layer[l];
    const int md = P.route_dec[l], b = P.budget[l];
    y.method = md;
    y.b = b;
    y.cap = d.cap[l];
    y.unit_off = d.unit_off[l];
    y.row_off = d.row_off[l];
    y.pre_method = P.route_pre[l];
    y.pre_slots = P.slots[l];
    y.pre_row_off = pre_off;
    pre_off += rows_per_layer(P, B, l);
    if (y.cap > 0 && (md == KVEV_H2O || md == KVEV_TOVA))
      dp.n_att += B * P.H_kv;
    else if (y.cap > 0)
      dp.n_cheap += B * P.H_kv;
    y.att_end = dp.n_att;
    y.cheap_end = dp.n_cheap;
    if (y.cap == 0) continue;
    if (md == KVEV_H2O || md == KVEV_TOVA) {
      y.r = md == KVEV_TOVA ? 0 : (P.h2o_recent < 0 ? b / 2 : P.h2o_recent);
      if (b < 1 || y.r >= b) return KVEV_EINVAL;  // at least one slot must be evictable
    } else if (md == KVEV_STREAMING) {
      if (P.sink < 0 || b <= P.sink) return KVEV_EINVAL;
      y.sink = P.sink;
      y.recent = P.recent < 0 ? b - P.sink : std::min(P.recent, b - P.sink);
    }
  }
  return KVEV_OK;
}

// Shared memory of the step kernel: the logits of the largest H2O/TOVA unit.
// Dynamic shared memory of a decode step: G rows of logits per slot, or one
// row (the new keys) when the attention is supplied.
size_t dec_smem(const kvev_plan& P, const DecLayout& d, bool supplied_attention = false) {
  int cap = 0;
  for (int l = 0; l < P.L; ++l)
    if (d.cap[l] > 0 && (P.route_dec[l] == KVEV_H2O || P.route_dec[l] == KVEV_TOVA))
      cap = std::max(cap, d.cap[l]);
  const size_t rows = supplied_attention ? 1 : static_cast<size_t>(P.G);
  return cap == 0 ? 0 : sizeof(float) * rows * (cap + 1);
}

void set_state_ptrs(DecodeParams& dp, const DecLayout& d, void* dec_K, void* dec_V, void* state) {
  uint8_t* sb = static_cast<uint8_t*>(state);
  dp.K = dec_K;
  dp.V = dec_V;
  dp.lens = reinterpret_cast<int32_t*>(sb + d.lens);
  dp.count = reinterpret_cast<int32_t*>(sb + d.count);
  dp.evicted = reinterpret_cast<int32_t*>(sb + d.evicted);
  dp.pos = reinterpret_cast<int32_t*>(sb + d.pos);
  dp.acc = reinterpret_cast<float*>(sb + d.acc);
  dp.done = reinterpret_cast<int32_t*>(sb + d.done);
}

}  // namespace

extern "C" int kvev_decode_query(const kvev_plan* plan, int B, int growth, int64_t* rows,
                                 size_t* state_bytes) {
  if (!plan) return KVEV_EINVAL;
  DecLayout d;
  const int rc = dec_layout(*plan, B, growth, d);
  if (rc != KVEV_OK) return rc;
  if (rows) *rows = d.rows;
  if (state_bytes) *state_bytes = d.total;
  return KVEV_OK;
}

extern "C" int kvev_decode_layer(const kvev_plan* plan, int B, int growth, int layer,
                                 int64_t* row_offset, int* cap, int* unit_offset) {
  if (!plan || layer < 0 || layer >= plan->L) return KVEV_EINVAL;
  DecLayout d;
  const int rc = dec_layout(*plan, B, growth, d);
  if (rc != KVEV_OK) return rc;
  if (row_offset) *row_offset = d.row_off[layer];
  if (cap) *cap = d.cap[layer];
  if (unit_offset) *unit_offset = d.unit_off[layer];
  return KVEV_OK;
}

extern "C" int kvev_decode_state_offsets(const kvev_plan* plan, int B, int growth, size_t* offsets) {
  if (!plan || !offsets) return KVEV_EINVAL;
  DecLayout d;
  const int rc = dec_layout(*plan, B, growth, d);
  if (rc != KVEV_OK) return rc;
  offsets[0] = d.lens;
  offsets[1] = d.count;
  offsets[2] = d.evicted;
  offsets[3] = d.pos;
  offsets[4] = d.acc;
  return KVEV_OK;
}

extern "C" int kvev_decode_init(kvev_plan* plan, int B, int growth, const void* pre_K,
                                const void* pre_V, const int32_t* pre_idx,
                                const int32_t* pre_count, const float* h2o_state,
                                const int32_t* lens_dev, void* dec_K, void* dec_V, void* dec_state,
                                void* stream) {
  if (!plan || B < 0) return KVEV_EINVAL;
  kvev_plan& P = *plan;
  DecLayout d;
  int rc = dec_layout(P, B, growth, d);
  if (rc != KVEV_OK) return rc;
  if (B == 0 || d.units == 0) return KVEV_OK;
  if (!pre_K || !pre_V || !pre_idx || !pre_count || !lens_dev || !dec_K || !dec_V || !dec_state)
    return KVEV_EINVAL;
  if (!aligned16(pre_K) || !aligned16(pre_V) || !aligned16(dec_K) || !aligned16(dec_V) ||
      (reinterpret_cast<uintptr_t>(dec_state) & 255u))
    return KVEV_EINVAL;
  DecodeParams dp;
  rc = dec_params(P, B, d, dp);
  if (rc != KVEV_OK) return rc;
  rc = ensure_device(plan);
  if (rc != KVEV_OK) return rc;
  set_state_ptrs(dp, d, dec_K, dec_V, dec_state);
  dp.status = P.ctx.status;
  dp.pre_K = pre_K;
  dp.pre_V = pre_V;
  dp.pre_idx = pre_idx;
  dp.pre_count = pre_count;
  dp.h2o_state = h2o_state;
  dp.lens_in = lens_dev;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  P.last_stream = s;
  return launch_decode_init(dp, s) == cudaSuccess ? KVEV_OK : KVEV_ECUDA;
}

namespace {

// One decode step; the H2O / TOVA layers take their attention from q_new
// (attn == nullptr) or from the caller (attn[l]).
int decode_step_impl(kvev_plan* plan, int B, int growth, void* dec_K, void* dec_V, void* dec_state,
                     const void* const* k_new, const void* const* v_new, const void* const* q_new,
                     const float* const* attn, void* stream) {
  if (!plan || B < 0) return KVEV_EINVAL;
  kvev_plan& P = *plan;
  DecLayout d;
  int rc = dec_layout(P, B, growth, d);
  if (rc != KVEV_OK) return rc;
  if (B == 0) return KVEV_OK;
  if (!dec_state || (reinterpret_cast<uintptr_t>(dec_state) & 255u)) return KVEV_EINVAL;
  if (d.units > 0) {
    if (!dec_K || !dec_V || !k_new || !v_new || (!q_new && !attn) || !aligned16(dec_K) ||
        !aligned16(dec_V))
      return KVEV_EINVAL;
    if (!decode_supported(P.d, P.G)) return KVEV_ENOTSUP;
  }
  DecodeParams dp;
  rc = dec_params(P, B, d, dp);
  if (rc != KVEV_OK) return rc;
  for (int l = 0; l < P.L; ++l) {
    if (d.cap[l] == 0) continue;
    if (!k_new[l] || !v_new[l] || !aligned16(k_new[l]) || !aligned16(v_new[l])) return KVEV_EINVAL;
    const bool attends = P.route_dec[l] == KVEV_H2O || P.route_dec[l] == KVEV_TOVA;
    if (attends && attn) {
      if (!attn[l] || (reinterpret_cast<uintptr_t>(attn[l]) & 3u)) return KVEV_EINVAL;
      dp.attn[l] = attn[l];
    } else if (attends && (!q_new[l] || !aligned16(q_new[l]))) {
      return KVEV_EINVAL;
    }
    dp.k_new[l] = k_new[l];
    dp.v_new[l] = v_new[l];
    dp.q_new[l] = q_new ? q_new[l] : nullptr;
  }
  rc = ensure_device(plan);
  if (rc != KVEV_OK) return rc;
  const size_t smem = dec_smem(P, d, attn != nullptr);
  if (smem + 1024 > static_cast<size_t>(P.ctx.smem_optin)) return KVEV_ENOTSUP;
  set_state_ptrs(dp, d, dec_K, dec_V, dec_state);
  dp.status = P.ctx.status;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  P.last_stream = s;
  return launch_decode_step(dp, smem, s) == cudaSuccess ? KVEV_OK : KVEV_ECUDA;
}

}  // namespace

extern "C" int kvev_decode_step(kvev_plan* plan, int B, int growth, void* dec_K, void* dec_V,
                                void* dec_state, const void* const* k_new,
                                const void* const* v_new, const void* const* q_new,
                                void* stream) {
  return decode_step_impl(plan, B, growth, dec_K, dec_V, dec_state, k_new, v_new, q_new, nullptr,
                          stream);
}

extern "C" int kvev_decode_step_attn(kvev_plan* plan, int B, int growth, void* dec_K, void* dec_V,
                                     void* dec_state, const void* const* k_new,
                                     const void* const* v_new, const float* const* attn,
                                     void* stream) {
  if (!attn) return KVEV_EINVAL;
  return decode_step_impl(plan, B, growth, dec_K, dec_V, dec_state, k_new, v_new, nullptr, attn,
                          stream);
}

// ---------------------------------------------------------------------------
// Prefill eviction without allocation: the workspace is a file-scope device
// array instead of caller memory.  Its name is only a host-side stand-in, so
// host code obtains the array's device address per device with
// cudaGetSymbolAddress (with that device current) and passes that pointer on.
// ---------------------------------------------------------------------------
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[KVEV_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

struct NoallocDevice {
  bool ready = false;
  DevCtx ctx;
  void* scratch = nullptr;  // device address of g_noalloc_scratch on this device
};

std::mutex g_noalloc_mu;
NoallocDevice g_noalloc[kMaxDevices];

}  // namespace

extern "C" int kvev_evict_prefill_noalloc(kvev_plan* plan, const void* const* K,
                                          const void* const* V, const void* const* Q_win,
                                          const int32_t* lens_dev, int B, int S_cap, void* out_K,
                                          void* out_V, int32_t* out_idx, int32_t* out_count,
                                          float* h2o_state, int32_t* device_status, void* stream) {
  // The status word is required: the scratch is shared by every call, so the
  // kernels' status bits can only reach the caller through its own word.
  if (!plan || B < 0 || S_cap < 1 || !device_status) return KVEV_EINVAL;
  if (reinterpret_cast<uintptr_t>(device_status) & 3u) return KVEV_EINVAL;
  kvev_plan& P = *plan;
  if (B == 0) return KVEV_OK;
  int rc = check_prefill_args(P, K, V, Q_win, nullptr, lens_dev, B, S_cap, out_K, out_V, out_idx,
                              out_count);
  if (rc != KVEV_OK) return rc;
  if (ws_layout(P, B, S_cap).total > KVEV_NOALLOC_SCRATCH_BYTES) return KVEV_ENOMEM;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KVEV_ECUDA;
  if (dev < 0 || dev >= kMaxDevices) return KVEV_ENOTSUP;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  NoallocDevice& nd = g_noalloc[dev];
  if (!nd.ready) {  // once per device, with that device current
    rc = query_device(nd.ctx, dev);
    if (rc != KVEV_OK) return rc;
    if (cudaGetSymbolAddress(&nd.scratch, g_noalloc_scratch) != cudaSuccess) return KVEV_ECUDA;
    nd.ready = true;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(device_status, 0, sizeof(int32_t), s) != cudaSuccess) return KVEV_ECUDA;
  nd.ctx.status = reinterpret_cast<int*>(device_status);
  P.last_stream = s;
  return evict_impl(P, nd.ctx, K, V, Q_win, nullptr, lens_dev, B, S_cap, out_K, out_V, out_idx,
                    out_count, h2o_state, nd.scratch, s);
}
