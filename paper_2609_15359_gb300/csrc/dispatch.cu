// dispatch.cu -- global memory-aware dispatch (Sec. 3.3, Algorithm 1).
//
// Horizon SNAPSHOT.  For candidate j with live steps u_j and decoder k the
// peak is p_j + 1 + M_k(u_j) with M_k(u) = max_{t<u}(K[k][t] + t): one prefix
// maximum per decoder, shared by every candidate.  Writing A_k(u) =
// cap_k - 1 - M_k(u), decoder k is feasible for j iff p_j <= A_k(u_j) and the
// headroom is A_k(u_j) - p_j.  The rule (smallest Q among feasible decoders,
// else largest headroom, ties to the lowest index) then needs, per horizon
// column u, only
//   * PMq_u[i] = max over the first i+1 decoders in (Q, index) order of
//     A_k(u): the first position where it reaches p_j is the chosen decoder;
//   * max_k A_k(u) and its lowest arg-max for the fallback.
// So K is read exactly once, tile by tile over the horizon, with all D rows of
// a tile staged in shared memory by one TMA copy; the carry of the prefix
// maximum across tiles is resolved by decoupled look-back; and each candidate
// costs a binary search over D instead of D scores.  Candidates are first
// bucketed by the tile of their last live step so each tile serves its own.
//
// SEQUENTIAL (reservation after each choice) and the literal Algorithm 1
// modes are separate kernels below.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>

#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kMaxD = 1024;
constexpr int kMainThreads = 512;
constexpr int kBoxRows = 256;  // TMA box height limit

// ---------------------------------------------------------------------------
// TMA / mbarrier primitives (inline PTX)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile(
      "{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n" ::"r"(
          smem_u32(bar)),
      "r"(bytes)
      : "memory");
}
__device__ __forceinline__ bool mbar_test_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for a barrier phase; false if the bound expired.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
  for (uint32_t spins = 0; !mbar_test_wait(bar, parity); ++spins) {
    if (spins > kSpinLimit) return false;
    __nanosleep(20);
  }
  return true;
}
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// ---------------------------------------------------------------------------
// SNAPSHOT preparation: bucket candidates by the horizon tile of u_j - 1.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int candidate_steps(int32_t U, int H) {
  return U < 1 ? 1 : (U > H ? H : U);
}

__global__ void bin_count_kernel(int64_t J, int H, int W2, const int32_t *__restrict__ cp,
                                 const int32_t *__restrict__ cb, uint32_t *tcount,
                                 int32_t *choice, int64_t *headroom, int32_t *status) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  bool bad = false;
  for (int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; j < J; j += stride) {
    const int32_t p = cp[j], U = cb[j];
    if ((p | U) < 0) {
      bad = true;
      choice[j] = -1;
      if (headroom) headroom[j] = 0;
      continue;
    }
    const int u = candidate_steps(U, H);
    atomicAdd(&tcount[(u - 1) / W2], 1u);
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
}

// Exclusive scan of the T2 tile counts into toff[0..T2] (single block).
__global__ void __launch_bounds__(1024) bin_scan_kernel(int T2, const uint32_t *tcount, uint32_t *toff) {
  __shared__ uint32_t s_warp[32];
  __shared__ uint32_t s_carry;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) s_carry = 0;
  __syncthreads();
  for (int base = 0; base < T2; base += 1024) {
    const int i = base + threadIdx.x;
    const uint32_t v = i < T2 ? tcount[i] : 0u;
    uint32_t incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    uint32_t wbase = 0;
    for (int w = 0; w < warp; ++w) wbase += s_warp[w];
    const uint32_t carry = s_carry;
    if (i < T2) toff[i] = carry + wbase + incl - v;
    __syncthreads();
    if (threadIdx.x == 1023) s_carry = carry + wbase + incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) toff[T2] = s_carry;
}

__global__ void bin_scatter_kernel(int64_t J, int H, int W2, const int32_t *__restrict__ cp,
                                   const int32_t *__restrict__ cb, const uint32_t *toff,
                                   uint32_t *tcursor, int32_t *ord) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; j < J; j += stride) {
    const int32_t p = cp[j], U = cb[j];
    if ((p | U) < 0) continue;
    const int tile = (candidate_steps(U, H) - 1) / W2;
    const uint32_t pos = toff[tile] + atomicAdd(&tcursor[tile], 1u);
    ord[pos] = static_cast<int32_t>(j);
  }
}

// ---------------------------------------------------------------------------
// SNAPSHOT main kernel: persistent, one CTA per SM, tiles taken in ticket
// order so that decoupled look-back always makes progress.
// ---------------------------------------------------------------------------
struct SnapArgs {
  int D, H, W2, T2, Drows, boxes, box_rows;  // Drows = rows per staged tile (>= D)
  int tile_stride;                           // elements per tile buffer (1 KB multiple)
  bool use_tma;
  const int32_t *K;
  const int32_t *cap, *Q, *cp, *cb;
  const uint32_t *toff;
  const int32_t *ord;
  uint32_t *flags;  // per tile: 0 none, 1 aggregate, 2 inclusive
  uint32_t *agg;    // [T2][D] tile row maxima of K + t
  uint32_t *inc;    // [T2][D] inclusive prefix maxima through the tile
  uint32_t *ticket;
  int32_t *choice;
  int64_t *headroom;
  int32_t *status;
};

constexpr uint32_t kFlagAgg = 1, kFlagInc = 2;

template <int W2>
__global__ void __launch_bounds__(kMainThreads, 1)
dispatch_snapshot_kernel(const __grid_constant__ CUtensorMap tmap, SnapArgs a) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const int D = a.D, H = a.H;
  const int tid = threadIdx.x, lane = tid & 31;
  const size_t tile_elems = static_cast<size_t>(a.tile_stride);
  uint32_t *kbuf0 = reinterpret_cast<uint32_t *>(smem);
  uint32_t *kbuf1 = kbuf0 + tile_elems;
  int32_t *pmq = reinterpret_cast<int32_t *>(kbuf1 + tile_elems);  // [D][W2] by Q-position
  int32_t *s_cap = pmq + static_cast<size_t>(D) * W2;
  int32_t *s_sig = s_cap + D;  // Q-position -> decoder
  uint32_t *s_carry = reinterpret_cast<uint32_t *>(s_sig + D);
  uint32_t *s_agg = s_carry + D;
  constexpr int nch = kMainThreads / W2;  // position chunks per column
  int32_t *s_chPM = reinterpret_cast<int32_t *>(s_agg + D);  // [nch][W2]
  int32_t *s_chK = s_chPM + nch * W2;
  int32_t *s_argA = s_chK + nch * W2;  // [W2]
  long long *s_chA = reinterpret_cast<long long *>(
      (reinterpret_cast<uintptr_t>(s_argA + W2) + 15) & ~uintptr_t(15));  // [nch][W2]
  long long *s_maxA = s_chA + nch * W2;                                   // [W2]
  uint64_t *s_bar = reinterpret_cast<uint64_t *>(s_maxA + W2);            // [2]
  __shared__ int s_tile, s_next, s_abort;
  __shared__ uint32_t s_flag;

  // --- setup: capacities, queue order (stable by index), barriers ---------
  bool bad = false;
  for (int k = tid; k < D; k += kMainThreads) {
    const int32_t c = a.cap[k], q = a.Q[k];
    if ((c | q) < 0) bad = true;
    s_cap[k] = c;
  }
  for (int k = tid; k < D; k += kMainThreads) {
    const int32_t qk = a.Q[k];
    int rank = 0;
    for (int k2 = 0; k2 < D; ++k2) {
      const int32_t q2 = a.Q[k2];
      rank += (q2 < qk) || (q2 == qk && k2 < k);
    }
    s_sig[rank] = k;
  }
  if (bad) flag_error(a.status, MAPS_E_RANGE);
  if (tid == 0) {
    s_abort = 0;
    if (a.use_tma) {
      mbar_init(&s_bar[0], 1);
      mbar_init(&s_bar[1], 1);
      fence_mbar_init();
    }
  }
  __syncthreads();

  // every box is credited in full, rows past D included (zero-filled)
  const uint32_t tile_bytes = static_cast<uint32_t>(a.boxes) * a.box_rows * W2 * 4u;
  auto issue = [&](int tile, uint32_t *buf, uint64_t *bar) {
    mbar_expect_tx(bar, tile_bytes);
    for (int b = 0; b < a.boxes; ++b)
      tma_load_2d(buf + static_cast<size_t>(b) * a.box_rows * W2, &tmap, bar, tile * W2, b * a.box_rows);
  };
  if (tid == 0) {
    const int t = static_cast<int>(atomicAdd(a.ticket, 1u));
    s_tile = t;
    if (a.use_tma && t < a.T2) issue(t, kbuf0, &s_bar[0]);
  }
  __syncthreads();

  int cur = s_tile;
  int buf = 0;
  uint32_t phase[2] = {0u, 0u};
  constexpr int seg = W2 / 16;  // cells per row segment; 16 segments per row
  const int items = ((D * 16 + kMainThreads - 1) / kMainThreads) * kMainThreads;

  while (cur < a.T2) {
    uint32_t *kb = buf ? kbuf1 : kbuf0;
    const int64_t t0 = static_cast<int64_t>(cur) * W2;
    // prefetch the next tile into the other buffer (it was released by the
    // __syncthreads that ended the previous iteration)
    if (tid == 0) {
      const int nx = static_cast<int>(atomicAdd(a.ticket, 1u));
      s_next = nx;
      if (a.use_tma && nx < a.T2) {
        fence_proxy_async();
        issue(nx, buf ? kbuf0 : kbuf1, &s_bar[buf ^ 1]);
      }
    }
    if (a.use_tma) {
      if (!mbar_wait_bounded(&s_bar[buf], phase[buf])) {
        if (tid == 0) flag_error(a.status, MAPS_E_TIMEOUT);
        s_abort = 1;
      }
      phase[buf] ^= 1u;
    } else {
      for (size_t e = tid; e < static_cast<size_t>(D) * W2; e += kMainThreads) {
        const int r = static_cast<int>(e / W2), c = static_cast<int>(e % W2);
        const int64_t t = t0 + c;
        kb[e] = t < H ? static_cast<uint32_t>(a.K[static_cast<int64_t>(r) * H + t]) : 0u;
      }
    }
    __syncthreads();
    if (s_abort) break;

    // --- in-tile prefix maximum of K + t along each row ---------------------
    bool neg = false;
    for (int it = tid; it < items; it += kMainThreads) {
      const int row = it >> 4, sg = it & 15;
      const bool live_row = row < D;
      uint32_t v[seg];
      uint32_t run = 0;
#pragma unroll
      for (int j = 0; j < seg; ++j) {
        const int c = sg * seg + j;
        const int64_t t = t0 + c;
        uint32_t x = 0;
        if (live_row && t < H) {
          const uint32_t raw = kb[static_cast<size_t>(row) * W2 + c];
          if (static_cast<int32_t>(raw) < 0) neg = true;
          x = raw + static_cast<uint32_t>(t);  // K + t < 2^32
        }
        run = x > run ? x : run;
        v[j] = run;
      }
      uint32_t incl = run;
#pragma unroll
      for (int off = 1; off < 16; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off, 16);
        if (sg >= off) incl = y > incl ? y : incl;
      }
      uint32_t excl = __shfl_up_sync(0xffffffffu, incl, 1, 16);
      if (sg == 0) excl = 0;
      if (live_row) {
#pragma unroll
        for (int j = 0; j < seg; ++j) {
          const uint32_t y = v[j] > excl ? v[j] : excl;
          kb[static_cast<size_t>(row) * W2 + sg * seg + j] = y;
        }
        if (sg == 15) s_agg[row] = incl;
      }
    }
    if (neg) flag_error(a.status, MAPS_E_RANGE);
    __syncthreads();

    // --- carry across tiles: decoupled look-back ---------------------------
    uint32_t *agg_row = a.agg + static_cast<size_t>(cur) * D;
    uint32_t *inc_row = a.inc + static_cast<size_t>(cur) * D;
    for (int k = tid; k < D; k += kMainThreads) {
      s_carry[k] = 0;
      if (cur == 0)
        inc_row[k] = s_agg[k];
      else
        agg_row[k] = s_agg[k];
    }
    __syncthreads();
    if (tid == 0) {
      __threadfence();
      st_release_u32(a.flags + cur, cur == 0 ? kFlagInc : kFlagAgg);
    }
    for (int p = cur - 1; p >= 0; --p) {
      if (tid == 0) {
        uint32_t f = 0, spins = 0;
        while ((f = ld_acquire_u32(a.flags + p)) == 0) {
          if (++spins > kSpinLimit) {
            flag_error(a.status, MAPS_E_TIMEOUT);
            f = kFlagInc;  // give up: use what is there
            break;
          }
          __nanosleep(32);
        }
        s_flag = f;
      }
      __syncthreads();
      const uint32_t f = s_flag;
      const uint32_t *src = (f == kFlagInc ? a.inc : a.agg) + static_cast<size_t>(p) * D;
      for (int k = tid; k < D; k += kMainThreads) {
        const uint32_t y = __ldcg(src + k);
        if (y > s_carry[k]) s_carry[k] = y;
      }
      __syncthreads();
      if (f == kFlagInc) break;
    }
    if (cur > 0) {
      for (int k = tid; k < D; k += kMainThreads) {
        const uint32_t x = s_agg[k], c = s_carry[k];
        inc_row[k] = x > c ? x : c;
      }
      __syncthreads();
      if (tid == 0) {
        __threadfence();
        st_release_u32(a.flags + cur, kFlagInc);
      }
    }

    // --- per column: queue-ordered prefix max of A, and arg-max of A --------
    {
      const int c = tid % W2, ch = tid / W2;
      const int per = (D + nch - 1) / nch;
      const int i_lo = ch * per, i_hi = min(D, i_lo + per);
      int32_t run = -1;
      long long bestA = LLONG_MIN;
      int bestK = 0x7fffffff;
      for (int i = i_lo; i < i_hi; ++i) {
        const int k = s_sig[i];
        const uint32_t m0 = kb[static_cast<size_t>(k) * W2 + c], cr = s_carry[k];
        const uint32_t M = m0 > cr ? m0 : cr;
        const long long A = static_cast<long long>(s_cap[k]) - 1 - static_cast<long long>(M);
        const int32_t a32 = A < -1 ? -1 : static_cast<int32_t>(A);
        run = a32 > run ? a32 : run;
        if (A > bestA || (A == bestA && k < bestK)) {
          bestA = A;
          bestK = k;
        }
      }
      s_chPM[ch * W2 + c] = run;
      s_chA[ch * W2 + c] = bestA;
      s_chK[ch * W2 + c] = bestK;
      __syncthreads();
      int32_t pre = -1;
      for (int c2 = 0; c2 < ch; ++c2) {
        const int32_t y = s_chPM[c2 * W2 + c];
        pre = y > pre ? y : pre;
      }
      run = pre;
      for (int i = i_lo; i < i_hi; ++i) {
        const int k = s_sig[i];
        const uint32_t m0 = kb[static_cast<size_t>(k) * W2 + c], cr = s_carry[k];
        const uint32_t M = m0 > cr ? m0 : cr;
        const long long A = static_cast<long long>(s_cap[k]) - 1 - static_cast<long long>(M);
        const int32_t a32 = A < -1 ? -1 : static_cast<int32_t>(A);
        run = a32 > run ? a32 : run;
        pmq[static_cast<size_t>(i) * W2 + c] = run;
      }
      if (ch == 0) {
        long long bA = LLONG_MIN;
        int bK = 0x7fffffff;
        for (int c2 = 0; c2 < nch; ++c2) {
          const long long A = s_chA[c2 * W2 + c];
          const int k = s_chK[c2 * W2 + c];
          if (A > bA || (A == bA && k < bK)) {
            bA = A;
            bK = k;
          }
        }
        s_maxA[c] = bA;
        s_argA[c] = bK;
      }
    }
    __syncthreads();

    // --- the candidates whose last live step falls in this tile -----------
    {
      const uint32_t lo = a.toff[cur], hi = a.toff[cur + 1];
      for (uint32_t pos = lo + tid; pos < hi; pos += kMainThreads) {
        const int j = a.ord[pos];
        const int32_t p = a.cp[j];
        const int u = candidate_steps(a.cb[j], H);
        const int c = static_cast<int>(u - 1 - t0);
        int k;
        long long h;
        if (pmq[static_cast<size_t>(D - 1) * W2 + c] < p) {
          k = s_argA[c];  // nothing feasible: most headroom
          h = s_maxA[c] - p;
        } else {
          int l = 0, r = D - 1;  // first queue position whose prefix reaches p
          while (l < r) {
            const int mid = (l + r) >> 1;
            if (pmq[static_cast<size_t>(mid) * W2 + c] >= p)
              r = mid;
            else
              l = mid + 1;
          }
          k = s_sig[l];
          h = static_cast<long long>(pmq[static_cast<size_t>(l) * W2 + c]) - p;
        }
        a.choice[j] = k;
        if (a.headroom) a.headroom[j] = h;
      }
    }
    __syncthreads();
    cur = s_next;
    buf ^= 1;
  }
  (void)lane;
  // The loop ends normally only on a ticket >= T2, for which nothing was
  // prefetched.  After an abort, wait (bounded) for a prefetch in flight so
  // no copy lands in shared memory after the block has exited.
  if (a.use_tma && s_abort && s_next < a.T2) mbar_wait_bounded(&s_bar[buf ^ 1], phase[buf ^ 1]);
}

// ---------------------------------------------------------------------------
// Selection order shared by the sequential kernels: feasible before
// infeasible; feasible by queue length, infeasible by largest headroom; then
// the lowest decoder index.
// ---------------------------------------------------------------------------
struct Pick {
  int inf;      // 0 feasible, 1 infeasible, 2 none yet
  long long v;  // Q (feasible) or -headroom (infeasible)
  int k;
  long long h;  // headroom
};
__device__ __forceinline__ bool better(const Pick &x, const Pick &y) {
  if (x.inf != y.inf) return x.inf < y.inf;
  if (x.v != y.v) return x.v < y.v;
  return x.k < y.k;
}
__device__ __forceinline__ Pick make_pick(long long h, int32_t q, int k) {
  Pick p;
  p.inf = h >= 0 ? 0 : 1;
  p.v = h >= 0 ? static_cast<long long>(q) : -h;
  p.k = k;
  p.h = h;
  return p;
}
__device__ __forceinline__ Pick shfl_pick(const Pick &x, int off) {
  Pick y;
  y.inf = __shfl_xor_sync(0xffffffffu, x.inf, off);
  y.v = __shfl_xor_sync(0xffffffffu, x.v, off);
  y.k = __shfl_xor_sync(0xffffffffu, x.k, off);
  y.h = __shfl_xor_sync(0xffffffffu, x.h, off);
  return y;
}
// Block-wide best; every thread gets the result.
__device__ Pick block_best(Pick mine, Pick *s_w) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const Pick y = shfl_pick(mine, off);
    if (better(y, mine)) mine = y;
  }
  if (lane == 0) s_w[warp] = mine;
  __syncthreads();
  Pick b = s_w[0];
  for (int w = 1; w < nw; ++w)
    if (better(s_w[w], b)) b = s_w[w];
  __syncthreads();
  return b;
}
__device__ __forceinline__ Pick no_pick() {
  Pick p;
  p.inf = 2;
  p.v = 0;
  p.k = 0x7fffffff;
  p.h = 0;
  return p;
}

// ---------------------------------------------------------------------------
// SEQUENTIAL horizon dispatch: one block walks the candidates in order,
// scores every decoder, commits the footprint at the chosen one.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024, 1)
dispatch_sequential_kernel(int D, int H, int32_t *K, const int32_t *cap, int32_t *Q, int64_t J,
                           const int32_t *cp, const int32_t *cb, int32_t *choice,
                           int64_t *headroom, int32_t *status) {
  __shared__ uint32_t s_M[kMaxD];
  __shared__ Pick s_w[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  bool bad = false;
  for (int k = tid; k < D; k += blockDim.x)
    if ((cap[k] | Q[k]) < 0) bad = true;
  for (int64_t i = tid; i < static_cast<int64_t>(D) * H; i += blockDim.x)
    if (K[i] < 0) bad = true;
  if (bad) flag_error(status, MAPS_E_RANGE);
  __syncthreads();
  for (int64_t j = 0; j < J; ++j) {
    const int32_t p = cp[j], U = cb[j];
    if ((p | U) < 0) {
      if (tid == 0) {
        flag_error(status, MAPS_E_RANGE);
        choice[j] = -1;
        if (headroom) headroom[j] = 0;
      }
      continue;
    }
    const int u = candidate_steps(U, H);
    for (int k = warp; k < D; k += nwarp) {
      const int32_t *row = K + static_cast<int64_t>(k) * H;
      uint32_t m = 0;
      for (int t = lane; t < u; t += 32) {
        const uint32_t x = static_cast<uint32_t>(row[t]) + static_cast<uint32_t>(t);
        m = x > m ? x : m;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const uint32_t y = __shfl_xor_sync(0xffffffffu, m, off);
        m = y > m ? y : m;
      }
      if (lane == 0) s_M[k] = m;
    }
    __syncthreads();
    Pick mine = no_pick();
    for (int k = tid; k < D; k += blockDim.x) {
      const long long h = static_cast<long long>(cap[k]) - (static_cast<long long>(p) + 1 + s_M[k]);
      const Pick c = make_pick(h, Q[k], k);
      if (better(c, mine)) mine = c;
    }
    const Pick b = block_best(mine, s_w);
    if (tid == 0) {
      choice[j] = b.k;
      if (headroom) headroom[j] = b.h;
      if (Q[b.k] == 0x7fffffff)
        flag_error(status, MAPS_E_RANGE);
      else
        Q[b.k] += 1;
    }
    // reserve the candidate's footprint at the chosen decoder
    int32_t *row = K + static_cast<int64_t>(b.k) * H;
    bool over = false;
    for (int t = tid; t < u; t += blockDim.x) {
      long long v = static_cast<long long>(row[t]) + p + t + 1;
      if (v > 0x7fffffffLL) {
        over = true;
        v = 0x7fffffffLL;
      }
      row[t] = static_cast<int32_t>(v);
    }
    if (over) flag_error(status, MAPS_E_RANGE);
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Algorithm 1, literal.  Budgets: B_eff = floor(cap/S) - blocks held or
// reserved by the ongoing requests.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
alg1_budget_kernel(int D, int S, const int64_t *res_off, int64_t R, const int32_t *prompt,
                   const int32_t *gen, const int32_t *bound, const int32_t *cap,
                   long long *B_eff, int32_t *status) {
  __shared__ long long s_red[8];
  const int k = blockIdx.x;
  int64_t lo = res_off[k], hi = res_off[k + 1];
  if (lo < 0 || hi < lo || hi > R) {
    if (threadIdx.x == 0) flag_error(status, MAPS_E_RANGE);
    lo = hi = 0;
  }
  long long held = 0;
  bool bad = false;
  for (int64_t r = lo + threadIdx.x; r < hi; r += blockDim.x) {
    const int32_t p = prompt[r], g = gen[r], U = bound[r];
    if ((p | g | U) < 0) {
      bad = true;
      continue;
    }
    const long long reserve = static_cast<long long>(U) > static_cast<long long>(g) + 1
                                  ? static_cast<long long>(U)
                                  : static_cast<long long>(g) + 1;
    held += (static_cast<long long>(p) + reserve + S - 1) / S;
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) held += __shfl_xor_sync(0xffffffffu, held, off);
  if ((threadIdx.x & 31) == 0) s_red[threadIdx.x >> 5] = held;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long tot = 0;
    for (int w = 0; w < 8; ++w) tot += s_red[w];
    B_eff[k] = static_cast<long long>(cap[k]) / S - tot;
  }
}

// SNAPSHOT: every block rebuilds the queue-ordered prefix maximum of B_eff
// (D <= 1024) and serves a slice of the candidates by binary search.
__global__ void __launch_bounds__(256)
alg1_snapshot_kernel(int D, int S, const long long *B_eff, const int32_t *cap, const int32_t *Q,
                     int64_t J, const int32_t *cp, const int32_t *cb, int32_t *choice,
                     int64_t *headroom, int32_t *status) {
  __shared__ long long s_B[kMaxD];
  __shared__ long long s_pm[kMaxD];
  __shared__ int s_sig[kMaxD];
  __shared__ long long s_maxB;
  __shared__ int s_argB;
  const int tid = threadIdx.x;
  bool bad = false;
  for (int k = tid; k < D; k += blockDim.x) {
    s_B[k] = B_eff[k];
    if ((cap[k] | Q[k]) < 0) bad = true;
    const int32_t qk = Q[k];
    int rank = 0;
    for (int k2 = 0; k2 < D; ++k2) {
      const int32_t q2 = Q[k2];
      rank += (q2 < qk) || (q2 == qk && k2 < k);
    }
    s_sig[rank] = k;
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
  __syncthreads();
  if (tid < 32) {
    // warp 0: prefix max in queue order and arg-max in index order
    const int per = (D + 31) / 32, lo = tid * per, hi = min(D, lo + per);
    long long run = LLONG_MIN, bB = LLONG_MIN;
    int bK = 0x7fffffff;
    for (int i = lo; i < hi; ++i) {
      const long long x = s_B[s_sig[i]];
      run = x > run ? x : run;
    }
    for (int k = lo; k < hi; ++k)
      if (s_B[k] > bB) {
        bB = s_B[k];
        bK = k;
      }
    long long incl = run;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, off);
      if (tid >= off) incl = y > incl ? y : incl;
    }
    long long excl = __shfl_up_sync(0xffffffffu, incl, 1);
    if (tid == 0) excl = LLONG_MIN;
    long long r2 = excl;
    for (int i = lo; i < hi; ++i) {
      const long long x = s_B[s_sig[i]];
      r2 = x > r2 ? x : r2;
      s_pm[i] = r2;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const long long yB = __shfl_xor_sync(0xffffffffu, bB, off);
      const int yK = __shfl_xor_sync(0xffffffffu, bK, off);
      if (yB > bB || (yB == bB && yK < bK)) {
        bB = yB;
        bK = yK;
      }
    }
    if (tid == 0) {
      s_maxB = bB;
      s_argB = bK;
    }
  }
  __syncthreads();
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  bool badc = false;
  for (int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + tid; j < J; j += stride) {
    const int32_t p = cp[j], U = cb[j];
    if ((p | U) < 0) {
      badc = true;
      choice[j] = -1;
      if (headroom) headroom[j] = 0;
      continue;
    }
    const long long need = (static_cast<long long>(p) + U + S - 1) / S;  // Eq. (feasibility)
    int k;
    long long h;
    if (s_pm[D - 1] < need) {
      k = s_argB;  // nothing feasible: argmax B_eff
      h = s_maxB - need;
    } else {
      int l = 0, r = D - 1;  // argmin Q over the feasible set
      while (l < r) {
        const int mid = (l + r) >> 1;
        if (s_pm[mid] >= need)
          r = mid;
        else
          l = mid + 1;
      }
      k = s_sig[l];
      h = s_B[k] - need;
    }
    choice[j] = k;
    if (headroom) headroom[j] = h;
  }
  if (badc) flag_error(status, MAPS_E_RANGE);
}

// SEQUENTIAL: one block; after each choice B_eff[k*] -= B_need, Q[k*] += 1.
__global__ void __launch_bounds__(1024, 1)
alg1_sequential_kernel(int D, int S, long long *B_eff, const int32_t *cap, int32_t *Q, int64_t J,
                       const int32_t *cp, const int32_t *cb, int32_t *choice, int64_t *headroom,
                       int32_t *status) {
  __shared__ long long s_B[kMaxD];
  __shared__ Pick s_w[32];
  const int tid = threadIdx.x;
  bool bad = false;
  for (int k = tid; k < D; k += blockDim.x) {
    s_B[k] = B_eff[k];
    if ((cap[k] | Q[k]) < 0) bad = true;
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
  __syncthreads();
  for (int64_t j = 0; j < J; ++j) {
    const int32_t p = cp[j], U = cb[j];
    if ((p | U) < 0) {
      if (tid == 0) {
        flag_error(status, MAPS_E_RANGE);
        choice[j] = -1;
        if (headroom) headroom[j] = 0;
      }
      continue;
    }
    const long long need = (static_cast<long long>(p) + U + S - 1) / S;
    Pick mine = no_pick();
    for (int k = tid; k < D; k += blockDim.x) {
      const Pick c = make_pick(s_B[k] - need, Q[k], k);
      if (better(c, mine)) mine = c;
    }
    const Pick b = block_best(mine, s_w);
    if (tid == 0) {
      choice[j] = b.k;
      if (headroom) headroom[j] = b.h;
      s_B[b.k] -= need;
      if (Q[b.k] == 0x7fffffff)
        flag_error(status, MAPS_E_RANGE);
      else
        Q[b.k] += 1;
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
struct SnapGeom {
  int box_rows, boxes, Drows, W2, T2, tile_stride;
  size_t smem;
};

SnapGeom snap_geom(int D, int H) {
  SnapGeom g;
  g.box_rows = D < kBoxRows ? D : kBoxRows;
  g.boxes = (D + g.box_rows - 1) / g.box_rows;
  g.Drows = g.boxes * g.box_rows;
  int w = 256;
  while (w > 16 && static_cast<long long>(w) * g.Drows > 16384) w >>= 1;
  g.W2 = w;
  g.T2 = static_cast<int>((static_cast<long long>(H) + w - 1) / w);
  const int nch = kMainThreads / w;
  g.tile_stride = (g.Drows * w + 255) / 256 * 256;       // 1 KB-aligned buffers
  size_t b = 2 * static_cast<size_t>(g.tile_stride) * 4; // two K tiles
  b += static_cast<size_t>(D) * w * 4;                  // pmq
  b += 4 * static_cast<size_t>(D) * 4;                  // cap, sig, carry, agg
  b += 2 * static_cast<size_t>(nch) * w * 4 + w * 4;    // chPM, chK, argA
  b += 16;                                              // alignment slack
  b += static_cast<size_t>(nch) * w * 8 + w * 8;        // chA, maxA
  b += 2 * 8;                                           // barriers
  g.smem = b;
  return g;
}

struct SnapWs {
  uint32_t *zero;  // tcount[T2], tcursor[T2], flags[T2], ticket
  uint32_t *toff;
  int32_t *ord;
  uint32_t *agg, *inc;
};

SnapWs carve_snap(Carve &c, int D, int T2, int64_t J) {
  SnapWs w;
  w.zero = c.take<uint32_t>(3 * static_cast<size_t>(T2) + 1);
  w.toff = c.take<uint32_t>(static_cast<size_t>(T2) + 1);
  w.ord = c.take<int32_t>(static_cast<size_t>(J > 0 ? J : 1));
  w.agg = c.take<uint32_t>(static_cast<size_t>(T2) * D);
  w.inc = c.take<uint32_t>(static_cast<size_t>(T2) * D);
  return w;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

constexpr int kMaxH = 1 << 28;

template <int W2>
int run_snapshot(int grid, size_t smem, cudaStream_t s, const CUtensorMap &tmap, const SnapArgs &a) {
  MAPS_TRY(cuda_ok(cudaFuncSetAttribute(dispatch_snapshot_kernel<W2>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(smem))));
  dispatch_snapshot_kernel<W2><<<grid, kMainThreads, smem, s>>>(tmap, a);
  return launch_ok();
}

int launch_snapshot(int D, int H, const int32_t *K, const int32_t *cap, const int32_t *Q, int64_t J,
                    const int32_t *cp, const int32_t *cb, int32_t *choice, int64_t *headroom,
                    void *ws, cudaStream_t s) {
  const SnapGeom g = snap_geom(D, H);
  if (g.smem + 1024 > static_cast<size_t>(max_smem_optin())) return MAPS_E_INVALID;
  Carve cv(ws);
  const SnapWs w = carve_snap(cv, D, g.T2, J);
  int32_t *status = status_word(ws);
  uint32_t *tcount = w.zero, *tcursor = w.zero + g.T2, *flags = w.zero + 2 * static_cast<size_t>(g.T2);
  uint32_t *ticket = w.zero + 3 * static_cast<size_t>(g.T2);
  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.zero, 0, (3 * static_cast<size_t>(g.T2) + 1) * 4, s)));
  const int sms = sm_count();
  const int gb = static_cast<int>(std::min<int64_t>((J + 255) / 256, 4LL * sms));
  bin_count_kernel<<<gb, 256, 0, s>>>(J, H, g.W2, cp, cb, tcount, choice, headroom, status);
  bin_scan_kernel<<<1, 1024, 0, s>>>(g.T2, tcount, w.toff);
  bin_scatter_kernel<<<gb, 256, 0, s>>>(J, H, g.W2, cp, cb, w.toff, tcursor, w.ord);
  MAPS_TRY(launch_ok());

  CUtensorMap tmap;
  std::memset(&tmap, 0, sizeof(tmap));
  bool use_tma = (H % 4 == 0) && aligned(K, 16);
  PFN_cuTensorMapEncodeTiled_v12000 enc = use_tma ? tensor_map_encoder() : nullptr;
  if (enc == nullptr) use_tma = false;
  if (use_tma) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(D)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(H) * 4};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(g.W2), static_cast<cuuint32_t>(g.box_rows)};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r = enc(&tmap, CU_TENSOR_MAP_DATA_TYPE_INT32, 2, const_cast<int32_t *>(K), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) use_tma = false;
  }
  SnapArgs a;
  a.D = D;
  a.H = H;
  a.W2 = g.W2;
  a.T2 = g.T2;
  a.Drows = use_tma ? g.Drows : D;
  a.boxes = g.boxes;
  a.box_rows = g.box_rows;
  a.tile_stride = g.tile_stride;
  a.use_tma = use_tma;
  a.K = K;
  a.cap = cap;
  a.Q = Q;
  a.cp = cp;
  a.cb = cb;
  a.toff = w.toff;
  a.ord = w.ord;
  a.flags = flags;
  a.agg = w.agg;
  a.inc = w.inc;
  a.ticket = ticket;
  a.choice = choice;
  a.headroom = headroom;
  a.status = status;
  const int grid = std::min(sms, g.T2);
  switch (g.W2) {
    case 16: return run_snapshot<16>(grid, g.smem, s, tmap, a);
    case 32: return run_snapshot<32>(grid, g.smem, s, tmap, a);
    case 64: return run_snapshot<64>(grid, g.smem, s, tmap, a);
    case 128: return run_snapshot<128>(grid, g.smem, s, tmap, a);
    default: return run_snapshot<256>(grid, g.smem, s, tmap, a);
  }
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_dispatch_workspace_size(int32_t mode, int32_t D, int32_t H, int64_t J) {
  using namespace maps;
  Carve c(nullptr);
  if (mode == MAPS_MODE_SNAPSHOT && D >= 1 && H >= 1 && H <= kMaxH) {
    const SnapGeom g = snap_geom(D, H);
    carve_snap(c, D, g.T2, J);
  } else if ((mode == MAPS_MODE_ALG1_SNAPSHOT || mode == MAPS_MODE_ALG1_SEQUENTIAL) && D >= 1) {
    c.take<long long>(static_cast<size_t>(D));
  }
  return c.bytes();
}

int maps_dispatch(int32_t mode, int32_t D, int32_t H, int32_t S, int32_t *K, const int32_t *cap,
                  int32_t *Q, const int64_t *res_off, int64_t R, const int32_t *prompt,
                  const int32_t *gen, const int32_t *bound, int64_t J, const int32_t *cand_prompt,
                  const int32_t *cand_bound, int32_t *choice_out, int64_t *headroom_out, void *ws,
                  size_t ws_bytes, void *stream) {
  using namespace maps;
  if (mode < MAPS_MODE_SNAPSHOT || mode > MAPS_MODE_ALG1_SEQUENTIAL) return MAPS_E_INVALID;
  if (D < 1 || D > kMaxD || J < 0 || J > 0x7fffffffLL || cap == nullptr || Q == nullptr)
    return MAPS_E_INVALID;
  if (J > 0 && (cand_prompt == nullptr || cand_bound == nullptr || choice_out == nullptr))
    return MAPS_E_INVALID;
  const bool horizon = mode == MAPS_MODE_SNAPSHOT || mode == MAPS_MODE_SEQUENTIAL;
  if (horizon && (H < 1 || H > kMaxH || K == nullptr)) return MAPS_E_INVALID;
  if (!horizon && (S < 1 || res_off == nullptr || R < 0 ||
                   (R > 0 && (prompt == nullptr || gen == nullptr || bound == nullptr))))
    return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_dispatch_workspace_size(mode, D, H, J)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  if (J == 0) return MAPS_OK;
  switch (mode) {
    case MAPS_MODE_SNAPSHOT:
      return launch_snapshot(D, H, K, cap, Q, J, cand_prompt, cand_bound, choice_out, headroom_out, ws, s);
    case MAPS_MODE_SEQUENTIAL:
      dispatch_sequential_kernel<<<1, 1024, 0, s>>>(D, H, K, cap, Q, J, cand_prompt, cand_bound,
                                                    choice_out, headroom_out, status);
      return launch_ok();
    default: {
      Carve cv(ws);
      long long *B_eff = cv.take<long long>(static_cast<size_t>(D));
      alg1_budget_kernel<<<D, 256, 0, s>>>(D, S, res_off, R, prompt, gen, bound, cap, B_eff, status);
      if (mode == MAPS_MODE_ALG1_SNAPSHOT) {
        const int grid = static_cast<int>(std::min<int64_t>((J + 255) / 256, 4LL * sm_count()));
        alg1_snapshot_kernel<<<grid, 256, 0, s>>>(D, S, B_eff, cap, Q, J, cand_prompt, cand_bound,
                                                  choice_out, headroom_out, status);
      } else {
        alg1_sequential_kernel<<<1, 1024, 0, s>>>(D, S, B_eff, cap, Q, J, cand_prompt, cand_bound,
                                                  choice_out, headroom_out, status);
      }
      return launch_ok();
    }
  }
}

}  // extern "C"
