// score_common.cuh -- device pieces shared by the window-score kernel and the
// whole-prompt H2O kernels: bounded mbarrier waits and the per-row / per-key
// exp2 arithmetic of the softmax warpgroups.
#pragma once
#include "kvev_internal.cuh"

namespace kvev {
namespace {

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

__device__ __forceinline__ float max32(const float (&v)[32]) {
  float t[11];
#pragma unroll
  for (int j = 0; j < 10; ++j) t[j] = fmax3(v[3 * j], v[3 * j + 1], v[3 * j + 2]);
  t[10] = fmaxf(v[30], v[31]);
  const float a = fmax3(t[0], t[1], t[2]), b = fmax3(t[3], t[4], t[5]);
  const float c = fmax3(t[6], t[7], t[8]), e = fmax3(t[9], t[10], a);
  return fmax3(b, c, e);
}

__device__ __forceinline__ float sum4x2(const float2 (&a)[4]) {
  const float2 s = fadd2(fadd2(a[0], a[1]), fadd2(a[2], a[3]));
  return s.x + s.y;
}

// Keys of a 32-key chunk that row position tr cannot see are set to -inf.
__device__ __forceinline__ void mask_chunk(float (&v)[32], int k0, int tr) {
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (k0 + i > tr) v[i] = -INFINITY;
}

// One sweep-1 unit for one row: online base-2 (max, sum) update over the
// thread's 64 keys (two 32-key halves), with one rescale of the running sum.
__device__ __forceinline__ void s1_chunk64(const float (&v0)[32], const float (&v1)[32], float c, float& m,
                                           float& z) {
  const float mnew = fmaxf(m, fmaxf(max32(v0), max32(v1)) * c);
  const float base = mnew == -INFINITY ? 0.f : mnew;
  const float zs = z * ex2_approx(m - base);  // m = -inf -> 0
  const float2 cc = make_float2(c, c), nb = make_float2(-base, -base);
  float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
#pragma unroll
  for (int i = 0; i < 32; i += 2) {
    const float2 t0 = ffma2(make_float2(v0[i], v0[i + 1]), cc, nb);
    const float2 t1 = ffma2(make_float2(v1[i], v1[i + 1]), cc, nb);
    a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(ex2_approx(t0.x), ex2_approx(t0.y)));
    a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(ex2_approx(t1.x), ex2_approx(t1.y)));
  }
  z = zs + sum4x2(a);
  m = mnew;
}

// One 32-row chunk of sweep 2 for this thread's key: sum of exp2(s*c - lse2_r)
// into four packed accumulators; nl = -lse2 of the chunk's rows (shared memory).
// Every row of the chunk counts for this key: no per-element checks.
__device__ __forceinline__ void s2_chunk_full(const uint32_t (&rr)[32], float c, const float* nl,
                                              float2 (&a)[4]) {
  const float2 cc = make_float2(c, c);
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 l4 = lds4(nl + i);
    const float2 t0 = ffma2(make_float2(__uint_as_float(rr[i]), __uint_as_float(rr[i + 1])), cc,
                            make_float2(l4.x, l4.y));
    const float2 t1 = ffma2(make_float2(__uint_as_float(rr[i + 2]), __uint_as_float(rr[i + 3])),
                            cc, make_float2(l4.z, l4.w));
    a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(ex2_approx(t0.x), ex2_approx(t0.y)));
    a[((i >> 1) + 1) & 3] =
        fadd2(a[((i >> 1) + 1) & 3], make_float2(ex2_approx(t1.x), ex2_approx(t1.y)));
  }
}

__device__ __forceinline__ float2 merge_ms(float2 a, float2 e) {  // (max, sum) in base 2
  if (e.x == -INFINITY) return a;
  if (a.x == -INFINITY) return e;
  const float m = fmaxf(a.x, e.x);
  return make_float2(m, a.y * ex2_approx(a.x - m) + e.y * ex2_approx(e.x - m));
}

}  // namespace
}  // namespace kvev
