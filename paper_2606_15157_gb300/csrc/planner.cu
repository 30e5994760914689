// planner.cu -- host side of the plan constructor (Sec. 3.2 and 3.3): the
// route profiles' statistics, the TopRank route of Eq. (policy_routing), and
// the allocation scores of Sec. 3.3.  Host code only; everything is computed
// in fp64.
#include <cmath>
#include <cstdint>
#include <cstring>

#include "../../include/kvev.h"

namespace {

bool prefill_op(int m) {
  return m == KVEV_FULL || m == KVEV_SNAPKV || m == KVEV_H2O || m == KVEV_STREAMING;
}
bool decode_op(int m) {
  return m == KVEV_FULL || m == KVEV_H2O || m == KVEV_TOVA || m == KVEV_STREAMING;
}

}  // namespace

extern "C" int kvev_profile_cosine(double* C_out, const float* h_full, const float* h_cand, int L, int R,
                                   int64_t D) {
  if (!C_out || !h_full || !h_cand || L <= 0 || R <= 0 || D <= 0) return KVEV_EINVAL;
  for (int l = 0; l < L; ++l) {
    const float* f = h_full + static_cast<int64_t>(l) * D;
    double ff = 0.0;
    for (int64_t i = 0; i < D; ++i) ff += static_cast<double>(f[i]) * f[i];
    if (!std::isfinite(ff) || ff <= 0.0) return KVEV_EINVAL;
    for (int r = 0; r < R; ++r) {
      const float* c = h_cand + (static_cast<int64_t>(r) * L + l) * D;
      double cc = 0.0, fc = 0.0;
      for (int64_t i = 0; i < D; ++i) {
        cc += static_cast<double>(c[i]) * c[i];
        fc += static_cast<double>(f[i]) * c[i];
      }
      if (!std::isfinite(cc) || !std::isfinite(fc) || cc <= 0.0) return KVEV_EINVAL;
      C_out[static_cast<int64_t>(l) * R + r] = fc / (std::sqrt(ff) * std::sqrt(cc));
    }
  }
  return KVEV_OK;
}

extern "C" int kvev_score_ppl(double* s_out, const double* ppl, double ppl_full, int L, int R) {
  if (!s_out || !ppl || L <= 0 || R <= 0 || !std::isfinite(ppl_full)) return KVEV_EINVAL;
  for (int l = 0; l < L; ++l) {
    double best = -INFINITY;
    for (int r = 0; r < R; ++r) {
      const double v = ppl[static_cast<int64_t>(l) * R + r];
      if (!std::isfinite(v)) return KVEV_EINVAL;
      best = std::fmax(best, v - ppl_full);
    }
    s_out[l] = best;
  }
  return KVEV_OK;
}

extern "C" int kvev_score_entropy(double* H_out, const float* A, int L, int64_t rows, int K) {
  if (!H_out || !A || L <= 0 || rows <= 0 || K <= 0) return KVEV_EINVAL;
  for (int l = 0; l < L; ++l) {
    double total = 0.0;
    for (int64_t q = 0; q < rows; ++q) {
      const float* p = A + (static_cast<int64_t>(l) * rows + q) * K;
      double h = 0.0, sum = 0.0;
      for (int k = 0; k < K; ++k) {
        const double v = p[k];
        if (!std::isfinite(v) || v < 0.0) return KVEV_EINVAL;
        sum += v;
        if (v > 0.0) h -= v * std::log(v);
      }
      if (std::fabs(sum - 1.0) > 1e-3) return KVEV_EINVAL;  // each row is a distribution
      total += h;
    }
    H_out[l] = total / static_cast<double>(rows);
  }
  return KVEV_OK;
}

extern "C" int kvev_route_toprank(int32_t* route_out, const double* g, int L, int R, const int32_t* ops,
                                  const uint8_t* covered, int higher_is_better) {
  if (!route_out || !g || !ops || L <= 0 || R <= 0) return KVEV_EINVAL;
  for (int r = 0; r < R; ++r)
    if (!prefill_op(ops[r]) && !decode_op(ops[r])) return KVEV_EINVAL;
  for (int l = 0; l < L; ++l) {
    int best = -1;
    double bv = 0.0;
    for (int r = 0; r < R; ++r) {
      const int64_t i = static_cast<int64_t>(l) * R + r;
      if (covered && !covered[i]) continue;
      const double v = g[i];
      if (!std::isfinite(v)) return KVEV_EINVAL;
      // strictly better only: equal statistics keep the operator listed first
      if (best < 0 || (higher_is_better ? v > bv : v < bv)) {
        best = r;
        bv = v;
      }
    }
    route_out[l] = best < 0 ? KVEV_FULL : ops[best];
  }
  return KVEV_OK;
}

extern "C" int kvev_route_install(int32_t* route_prefill, int32_t* route_decode, const int32_t* route, int L,
                                  int scope) {
  if (!route_prefill || !route_decode || !route || L <= 0) return KVEV_EINVAL;
  if (scope < KVEV_SCOPE_PREFILL || scope > KVEV_SCOPE_BOTH) return KVEV_EINVAL;
  const bool pre = scope & KVEV_SCOPE_PREFILL, dec = scope & KVEV_SCOPE_DECODE;
  for (int l = 0; l < L; ++l) {
    const int m = route[l];
    if ((pre && !prefill_op(m)) || (dec && !decode_op(m)) || (!prefill_op(m) && !decode_op(m)))
      return KVEV_EINVAL;
  }
  for (int l = 0; l < L; ++l) {
    route_prefill[l] = pre ? route[l] : KVEV_FULL;
    route_decode[l] = dec ? route[l] : KVEV_FULL;
  }
  return KVEV_OK;
}
