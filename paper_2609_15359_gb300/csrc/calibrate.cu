// calibrate.cu -- uncertainty-aware calibration (Sec. 3.2) on the GPU.
//
// q is the k-th smallest one-sided score s_i = max(0, L_i - Lhat_i) with
// k = ceil((1 - alpha)(n + 1)).  The scores are unsigned 32-bit (the
// difference of two int32 values clamped at 0 fits), so q is found by a radix
// select whose passes narrow a range [lo, lo + 2^w) known to hold rank k:
//   - the first pass histograms a monotone bucket of every score: scores below
//     1,024 have a bin each, larger ones a bin per (leading-bit position, next
//     7 bits), so a bin covers 1 value below 1,024 and 2^(e-7) values at
//     leading bit e;
//   - each later pass histograms the next (up to) 12 bits of s - lo for the
//     scores inside the range.
// A range of one value is q, so a quantile below 1,024 takes one pass and any
// quantile at most three.
// Calibration sets above 8,192 scores take one cooperative kernel: one block
// of 1,024 threads per multiprocessor, each thread holding up to eight scores
// and eight of the queries' predictions in registers.  A pass adds the
// blocks' shared histograms into a global one and waits at a bounded grid
// barrier; every block then scans the global counts and picks the same bin,
// so the next pass needs no other exchange.  Once the range is one value each
// thread writes its queries' bounds U = pred + q.  Smaller sets take one block
// (select_small_kernel).
#include <algorithm>

#include "maps_internal.cuh"
#include "maps_bench.h"

namespace maps {
namespace {

constexpr int kBins = 4096;
constexpr int kPasses = 3;
constexpr int kSelectThreads = 1024;
constexpr uint32_t kExactBins = 1024;  // scores below this have a bin each
constexpr int kMantBits = 7;           // bits after the leading one, first pass
constexpr int kStepBits = 12;          // bits per later pass
constexpr int kRegItems = 8;           // scores, and predictions, a thread keeps in registers

// Test aid (maps_test_calibrate_absent_block): a block of the fused kernel
// that returns at once (-1: none), so that the others' grid barrier runs out,
// and the polls a barrier wait makes before it gives up.
__device__ int32_t g_cal_absent_block = -1;
__device__ uint32_t g_cal_spins = kSpinLimit;

struct SelectState {
  unsigned long long hist[kPasses][kBins];  // global bin counts per pass
  GridBar bar;                              // the fused kernel's grid barrier
  int32_t q;                                // the quantile once selected (0 before)
};

__device__ __forceinline__ uint32_t score(int32_t L, int32_t P) {
  long long d = static_cast<long long>(L) - static_cast<long long>(P);
  return d > 0 ? static_cast<uint32_t>(d) : 0u;
}

// First-pass bin: non-decreasing in s, at most 1024 + 22 * 128 = 3,840 bins.
__device__ __forceinline__ int first_bin(uint32_t s) {
  if (s < kExactBins) return static_cast<int>(s);
  const int e = 31 - __clz(s);  // leading bit, 10..31
  return static_cast<int>(kExactBins) + ((e - 10) << kMantBits) +
         static_cast<int>((s >> (e - kMantBits)) & ((1u << kMantBits) - 1u));
}

// Item u * 4 + c of thread t (of T in the grid) is element 4 (t + u T) + c:
// two 128-bit words per array when both pointers allow it.
__device__ __forceinline__ void load_items(const int32_t *__restrict__ a, int64_t cnt, int64_t t,
                                           int64_t T, bool vec, int32_t v[kRegItems]) {
#pragma unroll
  for (int u = 0; u < kRegItems / 4; ++u) {
    const int64_t i4 = t + u * T, e0 = 4 * i4;
    if (vec && e0 + 4 <= cnt) {
      const int4 x = __ldg(reinterpret_cast<const int4 *>(a) + i4);
      v[4 * u] = x.x, v[4 * u + 1] = x.y, v[4 * u + 2] = x.z, v[4 * u + 3] = x.w;
    } else {
#pragma unroll
      for (int c = 0; c < 4; ++c) v[4 * u + c] = e0 + c < cnt ? __ldg(a + e0 + c) : 0;
    }
  }
}

// The fused select and bounds (n > kSmallN).  in_regs: n <= kRegItems x the
// grid's threads, so each thread's scores stay in registers across passes;
// otherwise every pass reads them again.  pred_in_regs likewise for the m
// predictions.
__global__ void __launch_bounds__(kSelectThreads, 1)
calibrate_fused_kernel(const int32_t *__restrict__ L, const int32_t *__restrict__ P, int64_t n,
                       unsigned long long k0, const int32_t *__restrict__ pred, int64_t m,
                       int32_t *__restrict__ out, SelectState *st, int32_t *q_dev_out,
                       int32_t *status, int in_regs, int pred_in_regs) {
  pdl_prologue();
  if (static_cast<int>(blockIdx.x) == g_cal_absent_block) return;  // test aid, normally -1
  __shared__ uint32_t sh[kBins];
  __shared__ unsigned long long s_warp[kSelectThreads / 32];
  __shared__ uint32_t s_lo;
  __shared__ int s_w;
  __shared__ unsigned long long s_k;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t T = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + tid;
  const bool pvec = (reinterpret_cast<uintptr_t>(pred) % 16 == 0) &&
                    (reinterpret_cast<uintptr_t>(out) % 16 == 0);
  const bool svec = (reinterpret_cast<uintptr_t>(L) % 16 == 0) &&
                    (reinterpret_cast<uintptr_t>(P) % 16 == 0);
  // the predictions do not depend on q: their loads overlap the select
  int32_t pv[kRegItems];
  if (pred_in_regs) load_items(pred, m, t, T, pvec, pv);
  uint32_t sv[kRegItems];
  if (in_regs) {
    int32_t a[kRegItems], b[kRegItems];
    load_items(L, n, t, T, svec, a);
    load_items(P, n, t, T, svec, b);
#pragma unroll
    for (int i = 0; i < kRegItems; ++i) sv[i] = score(a[i], b[i]);
  }

  uint32_t lo = 0;
  int wlog = 32;
  unsigned long long k = k0;
  for (int pass = 0; pass < kPasses && wlog > 0; ++pass) {
    for (int b = tid; b < kBins; b += blockDim.x) sh[b] = 0;
    __syncthreads();
    const int shift = wlog > kStepBits ? wlog - kStepBits : 0;
    // First pass: the zero scores (about half of a length residual's scores)
    // are counted by one ballot per warp and every other lane adds alone,
    // since its bin is a single value or a narrow range.  Later passes
    // aggregate the lanes of each bin with a match, as no bin of a range is
    // known to be hot.  Every lane of a warp calls this together.
    auto visit = [&](uint32_t s, bool valid) {
      if (pass == 0) {
        const int d = first_bin(s);
        const unsigned zeros = __ballot_sync(0xffffffffu, valid && d == 0);
        if (zeros && lane == __ffs(zeros) - 1) atomicAdd(&sh[0], static_cast<uint32_t>(__popc(zeros)));
        if (valid && d > 0) atomicAdd(&sh[d], 1u);
      } else {
        const uint32_t r = s - lo;  // wlog <= 24 here
        if (s < lo || r >= (1u << wlog)) valid = false;
        const int d = valid ? static_cast<int>(r >> shift) : -1;
        const unsigned peers = __match_any_sync(0xffffffffu, d);
        if (valid && lane == __ffs(peers) - 1)
          atomicAdd(&sh[d], static_cast<uint32_t>(__popc(peers)));
      }
    };
    if (in_regs) {
#pragma unroll
      for (int i = 0; i < kRegItems; ++i)
        visit(sv[i], 4 * (t + (i / 4) * T) + (i % 4) < n);
    } else {
      // whole blocks step together, so every lane of a warp visits
      for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x; 4 * base < n; base += T) {
        const int64_t i4 = base + tid;
        int32_t a[4], b[4];
        if (svec && 4 * i4 + 4 <= n) {
          const int4 x = __ldg(reinterpret_cast<const int4 *>(L) + i4);
          const int4 y = __ldg(reinterpret_cast<const int4 *>(P) + i4);
          a[0] = x.x, a[1] = x.y, a[2] = x.z, a[3] = x.w;
          b[0] = y.x, b[1] = y.y, b[2] = y.z, b[3] = y.w;
        } else {
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const bool ok = 4 * i4 + c < n;
            a[c] = ok ? __ldg(L + 4 * i4 + c) : 0;
            b[c] = ok ? __ldg(P + 4 * i4 + c) : 0;
          }
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) visit(score(a[c], b[c]), 4 * i4 + c < n);
      }
    }
    __syncthreads();
    // start each block's flush at a different bin so blocks do not collide
    const int rot = static_cast<int>((blockIdx.x * 97u) % kBins);
    for (int i = tid; i < kBins; i += blockDim.x) {
      const int b = (i + rot) & (kBins - 1);
      if (sh[b]) atomicAdd(&st->hist[pass][b], static_cast<unsigned long long>(sh[b]));
    }
    if (!grid_barrier(&st->bar, status, g_cal_spins)) return;

    // every block: the bin holding rank k inside the range (the same counts,
    // so the same bin in every block)
    constexpr int kPer = kBins / kSelectThreads;  // 4 consecutive bins per thread
    unsigned long long c[kPer], tot = 0;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      c[j] = __ldcg(&st->hist[pass][tid * kPer + j]);
      tot += c[j];
    }
    unsigned long long incl = tot;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    unsigned long long excl = incl - tot;
    for (int w = 0; w < warp; ++w) excl += s_warp[w];
    if (excl < k && k <= excl + tot) {
      unsigned long long cum = excl;
      int d = 0;
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        if (k <= cum + c[j]) {
          d = tid * kPer + j;
          break;
        }
        cum += c[j];
      }
      // the new range: the bin's values
      uint32_t nlo;
      int nw;
      if (pass == 0) {
        if (d < static_cast<int>(kExactBins)) {
          nlo = static_cast<uint32_t>(d);
          nw = 0;
        } else {
          const int e = 10 + ((d - static_cast<int>(kExactBins)) >> kMantBits);
          const uint32_t top = (1u << kMantBits) |
                               static_cast<uint32_t>((d - static_cast<int>(kExactBins)) &
                                                     ((1 << kMantBits) - 1));
          nlo = top << (e - kMantBits);
          nw = e - kMantBits;
        }
      } else {
        nlo = lo + (static_cast<uint32_t>(d) << shift);
        nw = shift;
      }
      s_lo = nlo;
      s_w = nw;
      s_k = k - cum;
    }
    __syncthreads();
    lo = s_lo;
    wlog = s_w;
    k = s_k;
    __syncthreads();  // s_lo, s_w, s_k and s_warp are written again next pass
  }
  // three passes always close the range: q = lo
  const bool q_ok = lo <= 0x7fffffffu;
  const int32_t q = q_ok ? static_cast<int32_t>(lo) : 0;
  if (blockIdx.x == 0 && tid == 0) {
    if (q_ok) {
      st->q = q;
      if (q_dev_out) *q_dev_out = q;
    } else {
      flag_error(status, MAPS_E_RANGE);
    }
  }
  // U = pred + q (Eq. conformal_upper), saturated and flagged above INT32_MAX
  bool bad = false;
  auto bound_of = [&](int32_t p) {
    long long u = static_cast<long long>(p) + q;
    if (u > 0x7fffffffLL) {
      bad = true;
      u = 0x7fffffffLL;
    }
    return static_cast<int32_t>(u);
  };
  if (pred_in_regs) {
#pragma unroll
    for (int u = 0; u < kRegItems / 4; ++u) {
      const int64_t i4 = t + u * T, e0 = 4 * i4;
      if (pvec && e0 + 4 <= m) {
        reinterpret_cast<int4 *>(out)[i4] =
            make_int4(bound_of(pv[4 * u]), bound_of(pv[4 * u + 1]), bound_of(pv[4 * u + 2]),
                      bound_of(pv[4 * u + 3]));
      } else {
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (e0 + c < m) out[e0 + c] = bound_of(pv[4 * u + c]);
      }
    }
  } else {
    for (int64_t i = t; i < m; i += T) out[i] = bound_of(__ldg(pred + i));
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
}

// U = pred + q.  Four bounds per thread (one 128-bit load and store when
// both arrays allow it).  The predictions are the caller's input: the grid
// before this one is a select kernel of the same call, which writes only the
// select state, and it starts only once every earlier grid has completed.  So
// the loads are issued before the wait on that grid and overlap its tail;
// only the quantile is read after it.
__global__ void __launch_bounds__(256)
bound_kernel(const int32_t *__restrict__ pred, int64_t m, const SelectState *st,
             int32_t *__restrict__ out, int32_t *status) {
  const int64_t i4 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int64_t i = i4 * 4;
  const bool vec = (reinterpret_cast<uintptr_t>(pred) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(out) % 16 == 0) && i + 4 <= m;
  int32_t v[4] = {0, 0, 0, 0};
  if (vec) {
    const int4 x = __ldg(reinterpret_cast<const int4 *>(pred) + i4);
    v[0] = x.x;
    v[1] = x.y;
    v[2] = x.z;
    v[3] = x.w;
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c) v[c] = i + c < m ? __ldg(pred + i + c) : 0;
  }
  pdl_prologue();
  if (i >= m) return;
  const long long q = *reinterpret_cast<const volatile int32_t *>(&st->q);
  bool bad = false;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    long long u = static_cast<long long>(v[c]) + q;  // Eq. (conformal_upper)
    if (u > 0x7fffffffLL) {
      if (i + c < m) bad = true;
      u = 0x7fffffffLL;
    }
    v[c] = static_cast<int32_t>(u);
  }
  if (vec) {
    *reinterpret_cast<int4 *>(out + i) = make_int4(v[0], v[1], v[2], v[3]);
  } else {
#pragma unroll
    for (int c = 0; c < 4; ++c)
      if (i + c < m) out[i + c] = v[c];
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
}

// Small calibration sets (n <= kSmallN): a three-digit (11, 11, 10 bits) radix select,
// run by one block over the scores held in shared memory, then the bounds of
// up to kSmallM queries by the same block: one launch instead of a memset and
// four.
constexpr int kSmallN = 8192;
constexpr int kSmallM = 8192;
constexpr int kSmallThreads = 1024;
constexpr int kBitonicN = 2048;  // up to this many scores are sorted outright
constexpr int kSmallBins = 2 * kSmallThreads;  // 11-bit digits, two bins per thread

__global__ void __launch_bounds__(kSmallThreads)
select_small_kernel(const int32_t *__restrict__ L, const int32_t *__restrict__ P, int n,
                    unsigned long long k, const int32_t *__restrict__ pred, int m_inblock,
                    int32_t *__restrict__ out, SelectState *st, int32_t *q_dev_out,
                    int32_t *status) {
  pdl_prologue();
  extern __shared__ uint32_t s[];  // the scores (kBitonicN or kSmallN words, as launched)
  __shared__ uint32_t hist[kSmallBins];
  __shared__ uint32_t s_warp[kSmallThreads / 32];
  __shared__ uint32_t s_pick[2];  // the chosen bin, the rank left inside it
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < n; i += kSmallThreads) s[i] = score(__ldg(L + i), __ldg(P + i));
  uint32_t prefix = 0;
  if (n <= kBitonicN) {
    // few scores: sort them (bitonic network, padded to a power of two with
    // the largest value) and take the k-th smallest
    int Pn = 1;
    while (Pn < n) Pn <<= 1;
    for (int i = n + tid; i < Pn; i += kSmallThreads) s[i] = 0xffffffffu;
    __syncthreads();
    for (int kk = 2; kk <= Pn; kk <<= 1)
      for (int j = kk >> 1; j > 0; j >>= 1) {
        for (int i = tid; i < Pn; i += kSmallThreads) {
          const int l = i ^ j;
          if (l > i) {
            const uint32_t x = s[i], y = s[l];
            if ((x > y) == ((i & kk) == 0)) {
              s[i] = y;
              s[l] = x;
            }
          }
        }
        __syncthreads();
      }
    prefix = s[k - 1];
  } else {
    unsigned long long kr = k;  // rank still to find among the scores matching prefix
    for (int pass = 0; pass < kPasses; ++pass) {
      const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
      const int bits = pass == 2 ? 10 : 11;
      const int prev = pass == 0 ? 32 : (pass == 1 ? 21 : 10);  // bits above this digit
      for (int b = tid; b < kSmallBins; b += kSmallThreads) hist[b] = 0;
      __syncthreads();
      for (int i = tid; i < n; i += kSmallThreads) {
        const uint32_t v = s[i];
        if (prev == 32 || (v >> prev) == prefix) atomicAdd(&hist[(v >> shift) & ((1u << bits) - 1)], 1u);
      }
      __syncthreads();
      // exclusive scan of the bins (two per thread), then the bin holding rank kr
      const uint32_t c0 = hist[2 * tid], c1 = hist[2 * tid + 1];
      const uint32_t tot = c0 + c1;
      uint32_t incl = tot;
  #pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      if (lane == 31) s_warp[warp] = incl;
      __syncthreads();
      uint32_t excl = incl - tot;
      for (int w = 0; w < warp; ++w) excl += s_warp[w];
      if (excl < kr && kr <= static_cast<unsigned long long>(excl) + tot) {
        const bool first = kr <= static_cast<unsigned long long>(excl) + c0;
        s_pick[0] = 2 * tid + (first ? 0 : 1);
        s_pick[1] = static_cast<uint32_t>(kr - excl - (first ? 0 : c0));
      }
      __syncthreads();
      prefix = (prefix << bits) | s_pick[0];
      kr = s_pick[1];
      __syncthreads();  // hist and s_pick are reused by the next pass
    }
  }
  if (prefix > 0x7fffffffu) {
    if (tid == 0) flag_error(status, MAPS_E_RANGE);
    return;
  }
  const int32_t q = static_cast<int32_t>(prefix);
  if (tid == 0) {
    st->q = q;
    if (q_dev_out) *q_dev_out = q;
  }
  bool bad = false;
  for (int i = tid; i < m_inblock; i += kSmallThreads) {
    const long long u = static_cast<long long>(__ldg(pred + i)) + q;  // Eq. (conformal_upper)
    bad |= u > 0x7fffffffLL;
    out[i] = static_cast<int32_t>(u > 0x7fffffffLL ? 0x7fffffffLL : u);
  }
  if (__syncthreads_or(bad) && tid == 0) flag_error(status, MAPS_E_RANGE);
}

// Blocks of the fused kernel that can be resident at once (its grid limit as
// a cooperative launch).
int64_t fused_grid() {
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, calibrate_fused_kernel, kSelectThreads,
                                                    0) != cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  return static_cast<int64_t>(per_sm) * sm_count();
}

inline int64_t conformal_rank(int64_t n, uint32_t alpha_ppm) {
  const int64_t num = static_cast<int64_t>(1000000u - alpha_ppm) * (n + 1);
  return (num + 999999) / 1000000;
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_calibrate_workspace_size(int64_t n, int64_t m) {
  (void)n;
  (void)m;
  maps::Carve c(nullptr);
  c.take<maps::SelectState>(1);
  return c.bytes();
}

int maps_calibrate(const int32_t *true_len, const int32_t *pred_len, int64_t n,
                   uint32_t alpha_ppm, const int32_t *query_pred, int64_t m,
                   int32_t *bound_out, int32_t *q_dev_out, int32_t *q_host_out,
                   void *ws, size_t ws_bytes, void *stream) {
  using namespace maps;
  if (n < 0 || n > (int64_t(1) << 40) || alpha_ppm == 0 || alpha_ppm >= 1000000u || m < 0)
    return MAPS_E_INVALID;
  if (n > 0 && (true_len == nullptr || pred_len == nullptr)) return MAPS_E_INVALID;
  if (m > 0 && (query_pred == nullptr || bound_out == nullptr)) return MAPS_E_INVALID;
  const int64_t k = conformal_rank(n, alpha_ppm);
  if (k > n) return MAPS_E_UNBOUNDED;  // the quantile is +infinity
  MAPS_TRY(check_ws(ws, ws_bytes, maps_calibrate_workspace_size(n, m)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Carve cv(ws);
  SelectState *st = cv.take<SelectState>(1);
  int32_t *status = status_word(ws);

  const unsigned long long kk = static_cast<unsigned long long>(k);
  if (n <= kSmallN) {
    const int mi = m <= kSmallM ? static_cast<int>(m) : 0;  // bounds in the same block
    launch_pdl(select_small_kernel, 1, kSmallThreads,
               (n <= kBitonicN ? kBitonicN : kSmallN) * sizeof(uint32_t), s, true_len, pred_len,
               static_cast<int>(n),
               kk, query_pred, mi, bound_out, st, q_dev_out, status);
    MAPS_TRY(launch_ok());
    if (m <= kSmallM) m = 0;
  } else {
    MAPS_TRY(cuda_ok(cudaMemsetAsync(st, 0, sizeof(SelectState), s)));
    // one block of 1,024 threads per multiprocessor (its registers allow
    // one), at least a 128-bit word of both arrays per thread, and enough
    // threads to hold the predictions in registers
    const int64_t per = static_cast<int64_t>(kRegItems) * kSelectThreads;
    const int64_t want = std::max<int64_t>({int64_t(1), (n + 4 * kSelectThreads - 1) / (4 * kSelectThreads),
                                            (m + per - 1) / per});
    const int64_t g = std::min<int64_t>(want, fused_grid());
    const int in_regs = n <= per * g ? 1 : 0;
    const int pred_in_regs = m <= per * g ? 1 : 0;
    MAPS_TRY(launch_coop(calibrate_fused_kernel, g, kSelectThreads, 0, s, true_len, pred_len, n, kk,
                         query_pred, m, bound_out, st, q_dev_out, status, in_regs, pred_in_regs));
    m = 0;  // the bounds are written by the same kernel
  }
  if (m > 0) {
    const int64_t gb = (m + 1023) / 1024;
    if (gb > 0x7fffffffLL) return MAPS_E_INVALID;
    launch_pdl(bound_kernel, static_cast<unsigned>(gb), 256, 0, s, query_pred, m, st, bound_out, status);
    MAPS_TRY(launch_ok());
  }
  if (q_host_out != nullptr) {
    MAPS_TRY(cuda_ok(cudaMemcpyAsync(q_host_out, &st->q, sizeof(int32_t), cudaMemcpyDeviceToHost, s)));
    return maps_check(ws, stream);
  }
  return MAPS_OK;
}

int maps_test_calibrate_absent_block(int32_t block, uint32_t spin_limit) {
  using namespace maps;
  const uint32_t spins = spin_limit == 0 ? kSpinLimit : spin_limit;
  MAPS_TRY(cuda_ok(cudaMemcpyToSymbol(g_cal_absent_block, &block, sizeof(block))));
  MAPS_TRY(cuda_ok(cudaMemcpyToSymbol(g_cal_spins, &spins, sizeof(spins))));
  return MAPS_OK;
}

}  // extern "C"
