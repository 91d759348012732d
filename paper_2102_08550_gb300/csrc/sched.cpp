// Host scheduler of the Oscars round: iteration ticks, Algorithm 1 and the
// local-step counts.  Integer arithmetic after one fp64 quantisation, so the
// result is bit-for-bit reproducible on any host.
//
// Paper: Problem Formulation (Eq. 1 wait time mod(T, t_i), Eq. 2 max wait,
// Eq. 3 barrier T* with the constraint floor(T/min t) - floor(T/max t) < M,
// tau_i = floor(T* / t_i)) and Algorithm 1 (scan T = max t, max t + 1, ...
// while the constraint holds; keep the T with the smallest max wait).
//
// Readings: speed factors s_i (larger = faster) become ticks
// t_i = max(1, floor(Q/s_i + 0.5)); the first T = max(t) is always a
// candidate; the constraint is strict; ties keep the smallest T; the capped
// search also stops once T > M * max(t) (with equal t_i the constraint never
// fails); the literal search has no cap and needs min(t) < max(t).
#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdint>
#include <vector>

#include "../../include/oscars.h"
#include "internal.h"

namespace oscars {

namespace {
// Upper bound on the number of barrier candidates either search may scan
// (each candidate costs n modulo operations).
constexpr int64_t kMaxCandidates = int64_t(1) << 32;
}  // namespace

int iteration_ticks(const double* speed, int n, int64_t Q, int64_t* t, const char** why) {
  if (!speed || !t || n < 1) { *why = "iteration_ticks: null pointer or n < 1"; return OSCARS_EINVAL; }
  if (Q == 0) Q = 1000;
  if (Q < 1) { *why = "ticks_per_unit must be >= 1"; return OSCARS_EINVAL; }
  for (int i = 0; i < n; ++i) {
    const double s = speed[i];
    if (!(s > 0.0) || !std::isfinite(s)) { *why = "speed factors must be finite and > 0"; return OSCARS_EINVAL; }
    const double v = std::floor(static_cast<double>(Q) / s + 0.5);
    if (!(v < 9.0e18)) { *why = "iteration time overflows int64"; return OSCARS_EINVAL; }
    t[i] = v < 1.0 ? 1 : static_cast<int64_t>(v);
  }
  return OSCARS_OK;
}

int schedule_solve(const int64_t* t, int n, int64_t M, int mode, int64_t* T_star,
                   int64_t* max_wait, int32_t* tau, const char** why) {
  if (!t || n < 1) { *why = "schedule: null t_iter or n < 1"; return OSCARS_EINVAL; }
  if (M < 1) { *why = "schedule: M must be >= 1"; return OSCARS_EINVAL; }
  if (mode != OSCARS_SEARCH_CAPPED && mode != OSCARS_SEARCH_LITERAL) { *why = "schedule: bad search mode"; return OSCARS_EINVAL; }
  int64_t tmin = INT64_MAX, tmax = 0;
  for (int i = 0; i < n; ++i) {
    if (t[i] < 1) { *why = "schedule: iteration times must be >= 1"; return OSCARS_EINVAL; }
    if (t[i] < tmin) tmin = t[i];
    if (t[i] > tmax) tmax = t[i];
  }
  // bound the scan before running it
  int64_t last;  // largest T the search can reach
  if (mode == OSCARS_SEARCH_CAPPED) {
    if (M > INT64_MAX / tmax) { *why = "schedule: M * max(t) overflows"; return OSCARS_EINVAL; }
    last = M * tmax;
  } else {
    if (tmin == tmax) { *why = "schedule: literal search never ends when all t_i are equal"; return OSCARS_EINVAL; }
    // floor(T/tmin) - floor(T/tmax) > T/tmin - T/tmax - 1 >= M once
    // T >= (M + 1) * tmin * tmax / (tmax - tmin)
    const long double bound = static_cast<long double>(M + 1) * tmin * tmax / (tmax - tmin) + 1.0L;
    if (bound > static_cast<long double>(INT64_MAX / 2)) { *why = "schedule: literal search too long"; return OSCARS_EINVAL; }
    last = static_cast<int64_t>(bound);
  }
  if (last - tmax > kMaxCandidates / n) { *why = "schedule: search range too large"; return OSCARS_EINVAL; }

  int64_t T = tmax, best_T = tmax, best_w = INT64_MAX;
  for (;;) {
    int64_t w = 0;                              // Eq. 2: max_j mod(T, t_j)
    for (int j = 0; j < n; ++j) {
      const int64_t r = T % t[j];               // Eq. 1
      if (r > w) w = r;
    }
    if (w < best_w) { best_w = w; best_T = T; } // first minimum
    ++T;
    if (!((T / tmin) - (T / tmax) < M)) break;  // constraint of Eq. 3
    if (mode == OSCARS_SEARCH_CAPPED && T > M * tmax) break;
  }
  if (T_star) *T_star = best_T;
  if (max_wait) *max_wait = best_w;
  if (tau) {
    for (int i = 0; i < n; ++i) {
      const int64_t v = best_T / t[i];
      if (v > INT32_MAX) { *why = "schedule: local-step count overflows int32"; return OSCARS_EINVAL; }
      tau[i] = static_cast<int32_t>(v);
    }
  }
  return OSCARS_OK;
}

void merge_weights(int rule, const int32_t* tau, int n, float* w) {
  if (rule == OSCARS_W_LOCALSTEPS) {
    double sum = 0.0;
    for (int i = 0; i < n; ++i) sum += static_cast<double>(tau[i]);
    for (int i = 0; i < n; ++i) w[i] = static_cast<float>(static_cast<double>(tau[i]) / sum);
  } else {
    const float u = static_cast<float>(1.0 / static_cast<double>(n));
    for (int i = 0; i < n; ++i) w[i] = u;
  }
}

}  // namespace oscars

extern "C" {

oscars_status oscars_iteration_ticks(const double* speed, int32_t n, int64_t ticks_per_unit,
                                     int64_t* t_iter) {
  const char* why = "";
  return static_cast<oscars_status>(oscars::iteration_ticks(speed, n, ticks_per_unit, t_iter, &why));
}

oscars_status oscars_schedule_solve(const int64_t* t_iter, int32_t n, int64_t M,
                                    int32_t search_mode, int64_t* T_star, int64_t* max_wait,
                                    int32_t* tau) {
  const char* why = "";
  return static_cast<oscars_status>(
      oscars::schedule_solve(t_iter, n, M, search_mode, T_star, max_wait, tau, &why));
}

oscars_status oscars_merge_weights(int32_t rule, const int32_t* tau, int32_t n, float* w) {
  if (!w || n < 1) return OSCARS_EINVAL;
  if (rule == OSCARS_W_LOCALSTEPS) {
    if (!tau) return OSCARS_EINVAL;
    for (int i = 0; i < n; ++i)
      if (tau[i] < 1) return OSCARS_EINVAL;
  } else if (rule != OSCARS_W_UNIFORM) {
    return OSCARS_EINVAL;
  }
  oscars::merge_weights(rule, tau, n, w);
  return OSCARS_OK;
}

oscars_status oscars_policy_local_steps(int32_t policy, const int64_t* t_iter, int32_t n, int64_t M,
                                        int32_t search_mode, int32_t I, int32_t* tau, int64_t* barrier) {
  if (!t_iter || !tau || n < 1) return OSCARS_EINVAL;
  for (int i = 0; i < n; ++i)
    if (t_iter[i] < 1) return OSCARS_EINVAL;
  if (policy == OSCARS_POLICY_OSCARS) {
    const char* why = "";
    int64_t T = 0;
    const int st = oscars::schedule_solve(t_iter, n, M, search_mode, &T, nullptr, tau, &why);
    if (st != OSCARS_OK) return static_cast<oscars_status>(st);
    if (barrier) *barrier = T;
    return OSCARS_OK;
  }
  int32_t k = 0;
  if (policy == OSCARS_POLICY_BSP) k = 1;
  else if (policy == OSCARS_POLICY_LOCAL_SGD) k = I;
  else return OSCARS_EINVAL;
  if (k < 1) return OSCARS_EINVAL;
  int64_t b = 0;   // last push: max_i k * t_i
  for (int i = 0; i < n; ++i) {
    if (t_iter[i] > INT64_MAX / k) return OSCARS_EINVAL;
    tau[i] = k;
    b = std::max(b, static_cast<int64_t>(k) * t_iter[i]);
  }
  if (barrier) *barrier = b;
  return OSCARS_OK;
}

oscars_status oscars_partition_sizes(const int64_t* weight, int32_t n, int64_t total, int64_t unit,
                                     int64_t* sizes) {
  if (!weight || !sizes || n < 1 || unit < 1 || total < 0) return OSCARS_EINVAL;
  const int64_t Q = total / unit;   // whole units to hand out
  unsigned __int128 wsum = 0;
  for (int i = 0; i < n; ++i) {
    if (weight[i] < 1) return OSCARS_EINVAL;
    wsum += static_cast<unsigned __int128>(weight[i]);
  }
  // Hamilton's apportionment: floors of the exact shares, the spare units to
  // the largest remainders (exact integer arithmetic; ties to the lower index)
  std::vector<unsigned __int128> rem(n);
  std::vector<int64_t> units(n);
  int64_t given = 0;
  for (int i = 0; i < n; ++i) {
    const unsigned __int128 num = static_cast<unsigned __int128>(Q) * static_cast<unsigned __int128>(weight[i]);
    units[i] = static_cast<int64_t>(num / wsum);
    rem[i] = num % wsum;
    given += units[i];
  }
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return rem[a] > rem[b]; });
  for (int64_t k = 0; k < Q - given; ++k) units[order[k]] += 1;
  for (int i = 0; i < n; ++i)
    if (units[i] < 1) return OSCARS_EINVAL;   // a worker would get no data
  for (int i = 0; i < n; ++i) sizes[i] = units[i] * unit;
  return OSCARS_OK;
}

oscars_status oscars_round_clusters(const int32_t* tau, int32_t n, int32_t max_clusters, int32_t* order,
                                    int32_t* first, int32_t* clusters) {
  if (!tau || !order || !first || !clusters || n < 1) return OSCARS_EINVAL;
  for (int i = 0; i < n; ++i)
    if (tau[i] < 1) return OSCARS_EINVAL;
  std::vector<int32_t> ord(n);
  for (int i = 0; i < n; ++i) ord[i] = i;
  std::stable_sort(ord.begin(), ord.end(), [&](int32_t x, int32_t y) { return tau[x] > tau[y]; });
  const int ncl = max_clusters > 0 && max_clusters < n ? max_clusters : n;
  // longest processing time first: each worker to the cluster with the least
  // work so far (a worker costs tau + 1/2: its steps and about half a step of
  // model load; half-integers are exact in a double)
  std::vector<std::vector<int32_t>> lists(ncl);
  std::vector<double> load(ncl, 0.0);
  for (int32_t w : ord) {
    int k = 0;
    for (int j = 1; j < ncl; ++j)
      if (load[j] < load[k]) k = j;
    lists[k].push_back(w);
    load[k] += tau[w] + 0.5;
  }
  int at = 0;
  first[0] = 0;
  for (int k = 0; k < ncl; ++k) {
    for (int32_t w : lists[k]) order[at++] = w;
    first[k + 1] = at;
  }
  *clusters = ncl;
  return OSCARS_OK;
}

const char* oscars_status_string(int32_t s) {
  switch (s) {
    case OSCARS_OK: return "OSCARS_OK";
    case OSCARS_EINVAL: return "OSCARS_EINVAL";
    case OSCARS_ENOMEM: return "OSCARS_ENOMEM";
    case OSCARS_ECUDA: return "OSCARS_ECUDA";
    case OSCARS_ESTATE: return "OSCARS_ESTATE";
    case OSCARS_ETIMEOUT: return "OSCARS_ETIMEOUT";
    case OSCARS_ENOTSUP: return "OSCARS_ENOTSUP";
    default: return "OSCARS_UNKNOWN";
  }
}

}  // extern "C"
