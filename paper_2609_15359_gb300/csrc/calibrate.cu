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
// quantile at most three.  The last block to finish a pass picks the bin that
// holds rank k; passes after the range has closed return at once.  Nothing
// returns to the host between passes.
#include <algorithm>

#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kBins = 4096;
constexpr int kPasses = 3;
constexpr int kSelectThreads = 1024;
constexpr uint32_t kExactBins = 1024;  // scores below this have a bin each
constexpr int kMantBits = 7;           // bits after the leading one, first pass
constexpr int kStepBits = 12;          // bits per later pass

struct SelectState {
  unsigned long long hist[kPasses][kBins];  // global bin counts per pass
  unsigned long long k_rem;                 // rank still to find inside the range
  uint32_t lo;                              // the range [lo, lo + 2^wlog) holding q
  int32_t wlog;
  uint32_t resolved;                        // set once the range is one value
  uint32_t done[kPasses];                   // blocks finished per pass
  int32_t q;                                // the quantile once selected
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

template <int PASS>
__global__ void __launch_bounds__(kSelectThreads)
select_pass_kernel(const int32_t *__restrict__ L, const int32_t *__restrict__ P,
                   int64_t n, unsigned long long k0, SelectState *st,
                   int32_t *q_dev_out, int32_t *status) {
  pdl_prologue();
  if (PASS > 0 && *reinterpret_cast<volatile uint32_t *>(&st->resolved)) return;
  __shared__ uint32_t sh[kBins];
  __shared__ int s_last;
  __shared__ unsigned long long s_warp[kSelectThreads / 32];

  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  // the range chosen so far and this pass's digit of s - lo
  const uint32_t lo = PASS == 0 ? 0u : *reinterpret_cast<volatile uint32_t *>(&st->lo);
  const int wlog = PASS == 0 ? 32 : *reinterpret_cast<volatile int32_t *>(&st->wlog);
  const int shift = wlog > kStepBits ? wlog - kStepBits : 0;

  // Histogram update.  First pass: the zero scores (about half of a length
  // residual's scores) are counted by one ballot per warp and every other lane
  // adds alone, since its bin is a single value or a narrow range.  Later
  // passes aggregate the lanes of each bin with a match, as no bin of a range
  // is known to be hot.
  const int lane = static_cast<int>(threadIdx.x & 31);
  auto visit = [&](uint32_t s, bool valid) {
    if constexpr (PASS == 0) {
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

  // Grid-stride loops whose bounds depend only on the block's first index,
  // so whole warps iterate together.
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t b0 = static_cast<int64_t>(blockIdx.x) * blockDim.x;
  const bool vec = (reinterpret_cast<uintptr_t>(L) % 16 == 0) &&
                   (reinterpret_cast<uintptr_t>(P) % 16 == 0);
  int64_t tail_start = 0;
  if (vec) {
    const int64_t n4 = n / 4;
    const int4 *L4 = reinterpret_cast<const int4 *>(L);
    const int4 *P4 = reinterpret_cast<const int4 *>(P);
    for (int64_t i0 = b0; i0 < n4; i0 += 4 * stride) {
      int4 a[4], b[4];
      bool ok[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {  // issue all loads first
        const int64_t i = i0 + u * stride + threadIdx.x;
        ok[u] = i < n4;
        a[u] = ok[u] ? __ldg(L4 + i) : make_int4(0, 0, 0, 0);
        b[u] = ok[u] ? __ldg(P4 + i) : make_int4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        visit(score(a[u].x, b[u].x), ok[u]);
        visit(score(a[u].y, b[u].y), ok[u]);
        visit(score(a[u].z, b[u].z), ok[u]);
        visit(score(a[u].w, b[u].w), ok[u]);
      }
    }
    tail_start = n4 * 4;
  }
  for (int64_t i0 = tail_start + b0; i0 < n; i0 += stride) {
    const int64_t i = i0 + threadIdx.x;
    const bool ok = i < n;
    visit(ok ? score(__ldg(L + i), __ldg(P + i)) : 0u, ok);
  }
  __syncthreads();

  // start each block's flush at a different bin so blocks do not collide
  const int rot = static_cast<int>((blockIdx.x * 97u) % kBins);
  for (int i = threadIdx.x; i < kBins; i += blockDim.x) {
    const int b = (i + rot) & (kBins - 1);
    if (sh[b]) atomicAdd(&st->hist[PASS][b], static_cast<unsigned long long>(sh[b]));
  }
  // one thread publishes the block's flush (the barrier orders every thread's
  // atomics before its fence, as a grid barrier does)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = (atomicAdd(&st->done[PASS], 1u) == gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // The last block: find the bin holding rank k inside the range.
  const unsigned long long k =
      PASS == 0 ? k0 : *reinterpret_cast<volatile unsigned long long *>(&st->k_rem);
  constexpr int kPer = kBins / kSelectThreads;  // 4 consecutive bins per thread
  unsigned long long c[kPer], tot = 0;
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    c[j] = __ldcg(&st->hist[PASS][threadIdx.x * kPer + j]);
    tot += c[j];
  }
  // exclusive scan of the per-thread totals
  const int warp = threadIdx.x >> 5;
  unsigned long long incl = tot;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    unsigned long long y = __shfl_up_sync(0xffffffffu, incl, off);
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
        d = threadIdx.x * kPer + j;
        break;
      }
      cum += c[j];
    }
    // the new range: the bin's values
    uint32_t nlo;
    int nw;
    if constexpr (PASS == 0) {
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
    st->lo = nlo;
    st->wlog = nw;
    st->k_rem = k - cum;
    if (nw == 0) {
      st->resolved = 1u;
      if (nlo > 0x7fffffffu) {
        flag_error(status, MAPS_E_RANGE);
      } else {
        st->q = static_cast<int32_t>(nlo);
        if (q_dev_out) *q_dev_out = static_cast<int32_t>(nlo);
      }
    }
  }
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
    // one block of 1,024 threads per multiprocessor (its registers allow one),
    // each reading at least a 128-bit word of both arrays per thread
    const int g = static_cast<int>(std::min<int64_t>(std::max<int64_t>(1, (n + 4 * kSelectThreads - 1) /
                                                                          (4 * kSelectThreads)),
                                                     sm_count()));
    launch_pdl(select_pass_kernel<0>, g, kSelectThreads, 0, s, true_len, pred_len, n, kk, st, q_dev_out, status);
    launch_pdl(select_pass_kernel<1>, g, kSelectThreads, 0, s, true_len, pred_len, n, kk, st, q_dev_out, status);
    launch_pdl(select_pass_kernel<2>, g, kSelectThreads, 0, s, true_len, pred_len, n, kk, st, q_dev_out, status);
    MAPS_TRY(launch_ok());
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

}  // extern "C"
