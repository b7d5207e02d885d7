/*
 * oracle_p.cpp -- the plain ("tier P") CPU oracle of the MAPS scheduler hot
 * path.
 *
 * TEST INFRASTRUCTURE ONLY: used by the test suite and by the benchmark's
 * CPU-baseline and reference legs, never by the product path.  It shares no
 * code with the CUDA library, nor with oracle.c, whose by-definition results
 * it must reproduce exactly (the tests check that).
 *
 * Where oracle.c writes each definition out step by step, this file computes
 * the same integers the plain way a CPU scheduler would:
 *   - quantile (Sec. 3.2, the rank after Eq. nonconformity): one selection
 *     (std::nth_element) for the k-th smallest score;
 *   - occupancy (App. A, Eq. kv_demand and Eq. admission over the horizon):
 *     per decoder, residents counted by their end step, then one pass down
 *     the horizon keeping the count and footprint sum of the residents still
 *     live, K(t) = sum + t * count;
 *   - SNAPSHOT dispatch (Sec. 3.3, Eq. feasibility and Algorithm 1): per
 *     decoder one forward pass for the prefix maximum of K(t) + t, so a
 *     (candidate, decoder) score is one lookup;
 *   - local order (Sec. 3.3, SJF by the bound with the maximum-waiting-time
 *     promotion): entries grouped by decoder, then each group sorted on its
 *     unique key.
 * Decoders, candidates and groups are independent, so each loop may run on
 * several host threads (OpenMP); the results do not depend on the thread
 * count.  No SIMD intrinsics.
 */
#include <algorithm>
#include <cstdint>
#include <cstdlib>
#include <vector>

#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

constexpr int64_t kI32Max = 2147483647LL;
constexpr int64_t kInfeasibleBase = int64_t(1) << 62;

enum { kOk = 0, kInvalid = -1, kRange = -2, kUnbounded = -3 };

int g_threads = 1;

int64_t rank_of(int64_t n, uint32_t alpha_ppm) {
  // ceil((1 - alpha)(n + 1)) with alpha in parts per million, exactly
  const int64_t num = static_cast<int64_t>(1000000u - alpha_ppm) * (n + 1);
  return (num + 999999) / 1000000;
}

bool offsets_ok(int32_t D, const int64_t *off, int64_t R) {
  if (off[0] < 0 || off[D] > R) return false;
  for (int32_t k = 0; k < D; ++k)
    if (off[k + 1] < off[k]) return false;
  return true;
}

}  // namespace

extern "C" {

// Host threads for the loops below (n <= 0: every core).  Returns the number
// that will be used (1 without OpenMP).
int oraclep_threads(int n) {
#ifdef _OPENMP
  g_threads = n > 0 ? n : omp_get_num_procs();
#else
  (void)n;
  g_threads = 1;
#endif
  return g_threads;
}

int oraclep_calibrate(const int32_t *true_len, const int32_t *pred_len, int64_t n,
                      uint32_t alpha_ppm, int64_t *q_out) {
  if (q_out == nullptr || n < 0 || n > (int64_t(1) << 40) || alpha_ppm == 0 ||
      alpha_ppm >= 1000000u || (n > 0 && (true_len == nullptr || pred_len == nullptr)))
    return kInvalid;
  const int64_t k = rank_of(n, alpha_ppm);
  if (k > n) return kUnbounded;
  std::vector<int64_t> s(static_cast<size_t>(n));
  for (int64_t i = 0; i < n; ++i) {
    const int64_t d = static_cast<int64_t>(true_len[i]) - pred_len[i];
    s[static_cast<size_t>(i)] = d > 0 ? d : 0;
  }
  std::nth_element(s.begin(), s.begin() + (k - 1), s.end());
  const int64_t q = s[static_cast<size_t>(k - 1)];
  if (q > kI32Max) return kRange;
  *q_out = q;
  return kOk;
}

int oraclep_bound(const int32_t *pred, int64_t m, int64_t q, int32_t *bound_out) {
  if (m < 0 || q < 0 || q > kI32Max || (m > 0 && (pred == nullptr || bound_out == nullptr)))
    return kInvalid;
  int status = kOk;
  for (int64_t i = 0; i < m; ++i) {
    int64_t u = static_cast<int64_t>(pred[i]) + q;  // Eq. (conformal_upper)
    if (u > kI32Max) {
      status = kRange;
      u = kI32Max;
    }
    bound_out[i] = static_cast<int32_t>(u);
  }
  return status;
}

int oraclep_occupancy(int32_t D, int32_t H, const int64_t *res_off, int64_t R,
                      const int32_t *prompt, const int32_t *gen, const int32_t *bound,
                      int32_t *K_out) {
  if (D < 1 || H < 1 || R < 0 || res_off == nullptr || K_out == nullptr ||
      (R > 0 && (prompt == nullptr || gen == nullptr || bound == nullptr)))
    return kInvalid;
  if (!offsets_ok(D, res_off, R)) return kRange;
  int status = kOk;
#pragma omp parallel num_threads(g_threads)
  {
    // per thread: residents ending at step e (exclusive), e in [1, H]
    std::vector<int64_t> cnt(static_cast<size_t>(H) + 1), sb(static_cast<size_t>(H) + 1);
    int local = kOk;
#pragma omp for schedule(dynamic, 1)
    for (int32_t k = 0; k < D; ++k) {
      std::fill(cnt.begin(), cnt.end(), 0);
      std::fill(sb.begin(), sb.end(), 0);
      for (int64_t r = res_off[k]; r < res_off[k + 1]; ++r) {
        if (prompt[r] < 0 || gen[r] < 0 || bound[r] < 0) {
          local = kRange;
          continue;
        }
        const int64_t b = static_cast<int64_t>(prompt[r]) + gen[r] + 1;
        int64_t e = static_cast<int64_t>(bound[r]) - gen[r];
        e = e < 1 ? 1 : (e > H ? H : e);
        cnt[static_cast<size_t>(e)] += 1;
        sb[static_cast<size_t>(e)] += b;
      }
      // down the horizon: at step t the live residents are those ending after t
      int64_t live = 0, sum = 0;
      int32_t *row = K_out + static_cast<int64_t>(k) * H;
      for (int64_t t = H - 1; t >= 0; --t) {
        live += cnt[static_cast<size_t>(t) + 1];
        sum += sb[static_cast<size_t>(t) + 1];
        int64_t v = sum + t * live;
        if (v > kI32Max) {
          local = kRange;
          v = kI32Max;
        }
        row[t] = static_cast<int32_t>(v);
      }
    }
    if (local != kOk) {
#pragma omp critical
      status = local;
    }
  }
  return status;
}

int oraclep_dispatch_snapshot(int32_t D, int32_t H, const int32_t *K, const int32_t *cap,
                              const int32_t *Q, int64_t J, const int32_t *cand_prompt,
                              const int32_t *cand_bound, int32_t *choice_out,
                              int64_t *headroom_out) {
  if (D < 1 || H < 1 || J < 0 || K == nullptr || cap == nullptr || Q == nullptr ||
      (J > 0 && (cand_prompt == nullptr || cand_bound == nullptr || choice_out == nullptr)))
    return kInvalid;
  // prefix maxima: pm[k][i] = max over t <= i of K[k][t] + t (kept between
  // calls, as a scheduler keeps its buffers)
  static std::vector<int64_t> pm;
  pm.resize(static_cast<size_t>(D) * H);
  int bad_k = 0;
#pragma omp parallel for num_threads(g_threads) schedule(static) reduction(| : bad_k)
  for (int32_t k = 0; k < D; ++k) {
    const int32_t *row = K + static_cast<int64_t>(k) * H;
    int64_t *out = pm.data() + static_cast<int64_t>(k) * H;
    int64_t m = INT64_MIN;
    for (int64_t t = 0; t < H; ++t) {
      if (row[t] < 0) bad_k = 1;
      const int64_t v = static_cast<int64_t>(row[t]) + t;
      m = v > m ? v : m;
      out[t] = m;
    }
  }
  if (bad_k) return kRange;
  int bad_c = 0;
#pragma omp parallel for num_threads(g_threads) schedule(static) reduction(| : bad_c)
  for (int64_t j = 0; j < J; ++j) {
    const int64_t p = cand_prompt[j], U = cand_bound[j];
    if (p < 0 || U < 0) {
      bad_c = 1;
      choice_out[j] = -1;
      if (headroom_out) headroom_out[j] = 0;
      continue;
    }
    const int64_t u = U < 1 ? 1 : (U > H ? H : U);
    int32_t best = -1;
    int64_t best_key = 0, best_h = 0;
    for (int32_t k = 0; k < D; ++k) {
      // peak of the footprint ramp p + t + 1 (t < u) over K: p + 1 + max(K + t)
      const int64_t h = static_cast<int64_t>(cap[k]) - (p + 1 + pm[static_cast<size_t>(k) * H + u - 1]);
      const int64_t key = h >= 0 ? static_cast<int64_t>(Q[k]) : kInfeasibleBase - h;
      if (best < 0 || key < best_key) {
        best = k;
        best_key = key;
        best_h = h;
      }
    }
    choice_out[j] = best;
    if (headroom_out) headroom_out[j] = best_h;
  }
  return bad_c ? kRange : kOk;
}

int oraclep_order_local(int64_t N, int32_t D, const int32_t *dec, const int32_t *bound,
                        const int32_t *wait, const int32_t *arrival, int32_t max_wait,
                        int32_t *perm_out, int64_t *seg_off_out) {
  if (N < 0 || N > kI32Max || D < 1 || seg_off_out == nullptr ||
      (N > 0 && (dec == nullptr || bound == nullptr || wait == nullptr || arrival == nullptr ||
                 perm_out == nullptr)))
    return kInvalid;
  for (int64_t i = 0; i < N; ++i)
    if (dec[i] < 0 || dec[i] >= D || bound[i] < 0 || arrival[i] < 0) return kRange;
  // group by decoder (a counting pass), then sort each group on its unique
  // key (not promoted, promoted ? arrival : bound, arrival, index)
  std::vector<int64_t> off(static_cast<size_t>(D) + 1, 0);
  for (int64_t i = 0; i < N; ++i) off[static_cast<size_t>(dec[i]) + 1] += 1;
  for (int32_t k = 0; k < D; ++k) off[static_cast<size_t>(k) + 1] += off[static_cast<size_t>(k)];
  std::vector<int64_t> cur(off.begin(), off.end() - 1);
  for (int64_t i = 0; i < N; ++i) perm_out[cur[static_cast<size_t>(dec[i])]++] = static_cast<int32_t>(i);
  struct Item {
    int64_t np, primary, arrival, idx;
  };
#pragma omp parallel num_threads(g_threads)
  {
    std::vector<Item> items;
#pragma omp for schedule(dynamic, 1)
    for (int32_t k = 0; k < D; ++k) {
      const int64_t a = off[static_cast<size_t>(k)], b = off[static_cast<size_t>(k) + 1];
      items.resize(static_cast<size_t>(b - a));
      for (int64_t s = a; s < b; ++s) {
        const int64_t i = perm_out[s];
        const bool promoted = wait[i] > max_wait;
        items[static_cast<size_t>(s - a)] = {promoted ? 0 : 1, promoted ? arrival[i] : bound[i],
                                             arrival[i], i};
      }
      std::sort(items.begin(), items.end(), [](const Item &x, const Item &y) {
        if (x.np != y.np) return x.np < y.np;
        if (x.primary != y.primary) return x.primary < y.primary;
        if (x.arrival != y.arrival) return x.arrival < y.arrival;
        return x.idx < y.idx;
      });
      for (int64_t s = a; s < b; ++s) perm_out[s] = static_cast<int32_t>(items[static_cast<size_t>(s - a)].idx);
    }
  }
  for (int32_t k = 0; k <= D; ++k) seg_off_out[k] = off[static_cast<size_t>(k)];
  return kOk;
}

}  // extern "C"
