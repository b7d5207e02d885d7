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
// So K is read at most once, tile by tile over the horizon (only the tiles
// holding some candidate's last live step), with all D rows of a tile staged
// in shared memory by one TMA copy; the carry of the prefix maximum into a
// tile comes from a per-decoder scan of the 16-step summary; per column the
// arg-max comes first, a candidate above every A_k is decided at once, and
// PMq is built only where some candidate fits, each of those then costing a
// binary search over D instead of D scores.  Candidates are first bucketed by
// the tile of their last live step so each tile serves its own.  Three
// launches: the carry scan and the bucket counts (independent, one launch),
// the bucket scatter, the scoring kernel.
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
#include "maps_bench.h"

namespace maps {
namespace {

constexpr int kMaxD = 1024;
constexpr int kMainThreads = 256;
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
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// ---------------------------------------------------------------------------
// SNAPSHOT preparation.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int candidate_steps(int32_t U, int H) {
  return U < 1 ? 1 : (U > H ? H : U);
}

constexpr int kSumBlock = 16;      // steps per kmax summary entry
constexpr int kUnitCands = 1024;   // candidates per work unit of the main kernel

// kmax[k][b] = max over the 16 steps of block b of K[k][t] + t, for callers
// that do not pass the summary from maps_project_occupancy.
__global__ void __launch_bounds__(256)
kmax_from_K_kernel(int D, int H, const int32_t *__restrict__ K, uint32_t *__restrict__ kmax,
                   int32_t *status) {
  pdl_prologue();
  const int64_t nb = (static_cast<int64_t>(H) + kSumBlock - 1) / kSumBlock;
  const int64_t total = nb * D;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  bool neg = false;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t k = i / nb, b = i - k * nb;
    const int32_t *row = K + k * H;
    const int64_t t0 = b * kSumBlock;
    uint32_t m = 0;
    for (int c = 0; c < kSumBlock; ++c) {
      const int64_t t = t0 + c;
      if (t >= H) break;
      const int32_t v = __ldg(row + t);
      if (v < 0) neg = true;
      const uint32_t x = static_cast<uint32_t>(v) + static_cast<uint32_t>(t);
      m = x > m ? x : m;
    }
    kmax[i] = m;
  }
  if (neg) flag_error(status, MAPS_E_RANGE);
}

// carry[k][i] = max of K[k][t] + t over t < i*W2 (0 for i = 0): the prefix
// maximum that horizon tile i inherits from the tiles before it.  One block
// per decoder; each thread reads 16 consecutive summary entries at once
// (whole tiles, as W2/16 divides 16), keeps its tiles' maxima in registers,
// and after a block scan writes its tiles' carries (the decoder's row of the
// carries is contiguous; a work unit later reads one word per decoder).
__device__ void carry_scan_block(int kk, int D, int H, int W2, int T2, const int32_t *__restrict__ K,
                                 bool check_kmax, const uint32_t *__restrict__ kmax,
                                 uint32_t *__restrict__ carry,
                                 const int32_t *__restrict__ Q, const int32_t *__restrict__ cap,
                                 int32_t *sig, int32_t *rank_of, int32_t *capq, int32_t *status) {
  __shared__ uint32_t s_w[8];
  __shared__ int s_rank;
  {
    // this decoder's position in (Q, index) order: the decoders before it
    const int32_t qk = __ldg(Q + kk);
    int r = 0;
    for (int k2 = threadIdx.x; k2 < D; k2 += blockDim.x) {
      const int32_t q2 = __ldg(Q + k2);
      r += (q2 < qk) || (q2 == qk && k2 < kk);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
    if (threadIdx.x == 0) s_rank = 0;
    __syncthreads();
    if ((threadIdx.x & 31) == 0) atomicAdd(&s_rank, r);
    __syncthreads();
    if (threadIdx.x == 0) {
      const int32_t ck = __ldg(cap + kk);
      if ((qk | ck) < 0) flag_error(status, MAPS_E_RANGE);
      sig[s_rank] = kk;
      rank_of[kk] = s_rank;
      capq[s_rank] = ck;
    }
  }
  constexpr int kPer = 16;
  const int k = kk;
  const int64_t nb = (static_cast<int64_t>(H) + kSumBlock - 1) / kSumBlock;
  const int bpt = W2 / kSumBlock;  // summary blocks per tile (1..16)
  const uint32_t *row = kmax + static_cast<int64_t>(k) * nb;
  uint32_t *out = carry + static_cast<int64_t>(k) * T2;  // carry[k][i], tile-contiguous per decoder
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool vec = (reinterpret_cast<uintptr_t>(row) % 16) == 0;
  uint32_t run = 0;
  for (int64_t c0 = 0; c0 < nb; c0 += 256 * kPer) {
    const int64_t b0 = c0 + threadIdx.x * kPer;
    uint32_t v[kPer];
    if (vec && b0 + kPer <= nb) {
#pragma unroll
      for (int q = 0; q < kPer; q += 4) {
        const uint4 x = __ldg(reinterpret_cast<const uint4 *>(row + b0 + q));
        v[q] = x.x, v[q + 1] = x.y, v[q + 2] = x.z, v[q + 3] = x.w;
      }
    } else {
#pragma unroll
      for (int q = 0; q < kPer; ++q) v[q] = b0 + q < nb ? __ldg(row + b0 + q) : 0u;
    }
    uint32_t m = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) m = v[q] > m ? v[q] : m;
    uint32_t incl = m;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl = y > incl ? y : incl;
    }
    if (lane == 31) s_w[warp] = incl;
    __syncthreads();
    uint32_t r = __shfl_up_sync(0xffffffffu, incl, 1);
    if (lane == 0) r = 0;
    uint32_t all = 0;
    for (int w = 0; w < 8; ++w) {
      if (w < warp) r = s_w[w] > r ? s_w[w] : r;
      all = s_w[w] > all ? s_w[w] : all;
    }
    r = r > run ? r : run;
    // this thread's tiles: [b0 / bpt, (b0 + kPer) / bpt)
    const int64_t tile0 = b0 / bpt;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      if (q % bpt == 0) {
        const int64_t ti = tile0 + q / bpt;
        if (ti < T2) out[ti] = r;
      }
      r = v[q] > r ? v[q] : r;
    }
    run = all > run ? all : run;
    __syncthreads();
  }
  if (check_kmax && threadIdx.x < 4) {
    // a caller's summary is compared with K at four blocks of this row (the
    // first, the last, the middle and one that varies with the decoder); a
    // mismatch there is reported, any other gives unspecified results
    const int64_t b = threadIdx.x == 0 ? 0 : threadIdx.x == 1 ? nb - 1 : threadIdx.x == 2 ? nb / 2
                                                                     : (k * 7919LL) % nb;
    const int32_t *kr = K + static_cast<int64_t>(k) * H;
    const int64_t t_end = (b + 1) * kSumBlock < H ? (b + 1) * kSumBlock : static_cast<int64_t>(H);
    long long mx = -1;
    for (int64_t t = b * kSumBlock; t < t_end; ++t) {
      const long long v = static_cast<long long>(__ldg(kr + t)) + t;
      mx = v > mx ? v : mx;
    }
    if (mx < 0 || static_cast<uint32_t>(mx) != __ldg(row + b)) flag_error(status, MAPS_E_INVALID);
  }
}

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Candidates are bucketed by the horizon tile holding their last live step
// u_j - 1.  When the tile count fits in shared memory each block first counts
// its candidates per tile locally and then adds one global count per
// non-empty tile; otherwise lanes with the same tile combine their atomic.
// Grid-stride loops run in whole warps.
constexpr int kBinSmem = 4096;

struct Unit {
  int32_t tile, start, count, pad;
};

__device__ void bin_scan_block(int T2, const uint32_t *tcount, uint32_t *toff, Unit *units,
                               uint32_t *nunits);

// Counting block b of nblk.
__device__ void bin_count_block(int b, int nblk, int64_t J, int H, int W2, int T2,
                                const int32_t *__restrict__ cp, const int32_t *__restrict__ cb,
                                uint32_t *tcount, int32_t *choice, int64_t *headroom,
                                int32_t *status, uint32_t *ticket, uint32_t *toff, Unit *units,
                                uint32_t *nunits) {
  __shared__ uint32_t s_h[kBinSmem];
  __shared__ bool s_last;
  const bool local = T2 <= kBinSmem;
  if (local)
    for (int i = threadIdx.x; i < T2; i += blockDim.x) s_h[i] = 0;
  __syncthreads();
  const int64_t stride = static_cast<int64_t>(nblk) * blockDim.x;
  bool bad = false;
  for (int64_t j0 = static_cast<int64_t>(b) * blockDim.x; j0 < J; j0 += stride) {
    const int64_t j = j0 + threadIdx.x;
    int tile = -1;
    if (j < J) {
      const int32_t p = cp[j], U = cb[j];
      if ((p | U) < 0) {
        bad = true;
        choice[j] = -1;
        if (headroom) headroom[j] = 0;
      } else {
        tile = (candidate_steps(U, H) - 1) / W2;
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, tile);
    if (tile >= 0 && (threadIdx.x & 31) == __ffs(peers) - 1)
      atomicAdd(local ? &s_h[tile] : &tcount[tile], static_cast<uint32_t>(__popc(peers)));
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
  if (local) {
    __syncthreads();
    // start each block's flush at a different tile so blocks do not collide
    const int rot = static_cast<int>((static_cast<int64_t>(b) * 97) % T2);
    for (int i = threadIdx.x; i < T2; i += blockDim.x) {
      const int t = (i + rot) % T2;
      if (s_h[t]) atomicAdd(&tcount[t], s_h[t]);
    }
  }
  // the last block to finish turns the counts into offsets and work units
  // (one thread publishes the block's counts: the barrier orders every
  // thread's atomics before its fence, as a grid barrier does)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(ticket, 1u) == static_cast<uint32_t>(nblk) - 1;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    bin_scan_block(T2, tcount, toff, units, nunits);
  }
}

// The two independent first steps in one launch: blocks [0, D) scan the
// carries of decoder blockIdx.x, the others count the candidates per tile.
__global__ void __launch_bounds__(256)
dispatch_prep_kernel(int ncarry, int D, int H, int W2, int T2, const int32_t *__restrict__ K,
                     bool check_kmax, const uint32_t *__restrict__ kmax,
                     uint32_t *__restrict__ carry, const int32_t *__restrict__ Q,
                     const int32_t *__restrict__ cap, int32_t *sig, int32_t *rank_of,
                     int32_t *capq, int64_t J, const int32_t *__restrict__ cp,
                     const int32_t *__restrict__ cb, uint32_t *tcount, int32_t *choice,
                     int64_t *headroom, int32_t *status, uint32_t *ticket, uint32_t *toff,
                     Unit *units, uint32_t *nunits) {
  pdl_prologue();
  if (static_cast<int>(blockIdx.x) < ncarry)
    carry_scan_block(blockIdx.x, D, H, W2, T2, K, check_kmax, kmax, carry, Q, cap, sig, rank_of,
                     capq, status);
  else
    bin_count_block(blockIdx.x - ncarry, gridDim.x - ncarry, J, H, W2, T2, cp, cb, tcount, choice,
                    headroom, status, ticket, toff, units, nunits);
}

// Run by the last counting block (any multiple of 32 threads up to 1024):
// tile offsets toff[0..T2] and the work units (a tile with c candidates gives
// ceil(c / kUnitCands) units; the unit count goes to *nunits).
__device__ void bin_scan_block(int T2, const uint32_t *tcount, uint32_t *toff, Unit *units,
                               uint32_t *nunits) {
  __shared__ uint32_t s_w[2][32];
  const int nt = blockDim.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // each thread takes a contiguous run of tiles: one block scan in all
  const int per = (T2 + nt - 1) / nt;
  const int i0 = min(T2, static_cast<int>(threadIdx.x) * per), i1 = min(T2, i0 + per);
  uint32_t sc = 0, su = 0;
  for (int i = i0; i < i1; ++i) {
    const uint32_t c = __ldcg(tcount + i);
    sc += c;
    su += (c + kUnitCands - 1) / kUnitCands;
  }
  uint32_t ic = sc, iu = su;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t yc = __shfl_up_sync(0xffffffffu, ic, off);
    const uint32_t yu = __shfl_up_sync(0xffffffffu, iu, off);
    if (lane >= off) {
      ic += yc;
      iu += yu;
    }
  }
  if (lane == 31) {
    s_w[0][warp] = ic;
    s_w[1][warp] = iu;
  }
  __syncthreads();
  uint32_t rc = ic - sc, ru = iu - su;  // exclusive starts of this thread's run
  for (int w = 0; w < warp; ++w) {
    rc += s_w[0][w];
    ru += s_w[1][w];
  }
  for (int i = i0; i < i1; ++i) {
    const uint32_t c = __ldcg(tcount + i);
    const uint32_t nu = (c + kUnitCands - 1) / kUnitCands;
    toff[i] = rc;
    for (uint32_t q = 0; q < nu; ++q) {
      Unit un;
      un.tile = i;
      un.start = static_cast<int32_t>(rc + q * kUnitCands);
      un.count = static_cast<int32_t>(min(static_cast<uint32_t>(kUnitCands), c - q * kUnitCands));
      un.pad = 0;
      units[ru + q] = un;
    }
    rc += c;
    ru += nu;
  }
  if (threadIdx.x == nt - 1) {  // the last thread's run ends at the totals
    toff[T2] = rc;
    *nunits = ru;
  }
}

// Place every valid candidate into its tile's bucket as (index, prompt,
// steps).  The order inside a bucket does not matter: each candidate's
// decision depends only on itself.
__global__ void __launch_bounds__(256)
bin_scatter_kernel(int64_t J, int H, int W2, int T2, const int32_t *__restrict__ cp,
                   const int32_t *__restrict__ cb, const uint32_t *toff, uint32_t *tcursor,
                   int32_t *ord, int32_t *sp, int32_t *su) {
  // The candidates are the caller's input and the grid before this one (the
  // counting kernel of the same call) writes only the workspace and the
  // call's outputs; it starts only once every earlier grid has completed.  So
  // this thread's first candidate is loaded before the wait on it.
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t b0 = static_cast<int64_t>(blockIdx.x) * blockDim.x;
  const int64_t j_first = b0 + threadIdx.x;
  const int32_t p_first = j_first < J ? cp[j_first] : -1;
  const int32_t u_first = j_first < J ? cb[j_first] : -1;
  pdl_prologue();
  __shared__ uint32_t s_h[kBinSmem];  // local counts, then local cursors
  __shared__ uint32_t s_b[kBinSmem];  // this block's base inside each bucket
  const bool local = T2 <= kBinSmem;
  if (local) {
    for (int i = threadIdx.x; i < T2; i += blockDim.x) s_h[i] = 0;
    __syncthreads();
    for (int64_t j0 = b0; j0 < J; j0 += stride) {
      const int64_t j = j0 + threadIdx.x;
      int tile = -1;
      if (j < J) {
        const int32_t U = j0 == b0 ? u_first : cb[j];
        if (((j0 == b0 ? p_first : cp[j]) | U) >= 0) tile = (candidate_steps(U, H) - 1) / W2;
      }
      const unsigned peers = __match_any_sync(0xffffffffu, tile);
      if (tile >= 0 && (threadIdx.x & 31) == __ffs(peers) - 1)
        atomicAdd(&s_h[tile], static_cast<uint32_t>(__popc(peers)));
    }
    __syncthreads();
    const int rot = static_cast<int>((static_cast<int64_t>(blockIdx.x) * 97) % T2);
    for (int i = threadIdx.x; i < T2; i += blockDim.x) {
      const int t = (i + rot) % T2;
      const uint32_t c = s_h[t];
      s_b[t] = c ? toff[t] + atomicAdd(&tcursor[t], c) : 0u;
      s_h[t] = 0;
    }
    __syncthreads();
  }
  for (int64_t j0 = b0; j0 < J; j0 += stride) {
    const int64_t j = j0 + threadIdx.x;
    int tile = -1, u = 0;
    int32_t p = 0;
    if (j < J) {
      p = j0 == b0 ? p_first : cp[j];
      const int32_t U = j0 == b0 ? u_first : cb[j];
      if ((p | U) >= 0) {
        u = candidate_steps(U, H);
        tile = (u - 1) / W2;
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, tile);
    const int leader = __ffs(peers) - 1;
    uint32_t base = 0;
    if (tile >= 0 && (threadIdx.x & 31) == leader) {
      const uint32_t c = static_cast<uint32_t>(__popc(peers));
      base = local ? s_b[tile] + atomicAdd(&s_h[tile], c) : toff[tile] + atomicAdd(&tcursor[tile], c);
    }
    base = __shfl_sync(0xffffffffu, base, leader);
    if (tile >= 0) {
      const uint32_t pos = base + __popc(peers & lanemask_lt());
      ord[pos] = static_cast<int32_t>(j);
      sp[pos] = p;
      su[pos] = u;
    }
  }
}

// ---------------------------------------------------------------------------
// SNAPSHOT main kernel: one CTA per work unit, a unit being (tile, a slice of
// the tile's candidates).  Tiles without candidates are never read: their
// contribution reaches later tiles through the carry, built from the summary.
// Several CTAs share an SM, so one CTA's TMA wait overlaps another's work.
// ---------------------------------------------------------------------------
struct SnapArgs {
  int D, H, W2, T2, Drows, boxes, box_rows;  // Drows = rows per staged tile (>= D)
  int tile_stride;                           // elements of the tile buffer (1 KB multiple)
  int comp_off;                              // words from the tile buffer to comp
  int region;                                // words from the tile buffer to the small arrays
  bool alias;                                // comp overwrites the tile (one row per thread)
  bool use_tma;
  const int32_t *K;
  const int32_t *sig, *rank_of, *capq;  // queue order
  const uint32_t *carry;                // [D][T2]
  const Unit *units;
  const uint32_t *nunits;
  const int32_t *ord, *sp, *su;
  int32_t *choice;
  int64_t *headroom;
  int32_t *status;
};

template <int W2>
__global__ void __launch_bounds__(kMainThreads, 4)
dispatch_snapshot_kernel(const __grid_constant__ CUtensorMap tmap, SnapArgs a) {
  pdl_prologue();
  extern __shared__ __align__(1024) unsigned char smem[];
  const int unit = blockIdx.x;
  if (unit >= static_cast<int>(*a.nunits)) return;
  const int D = a.D, H = a.H;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarpsM = kMainThreads / 32;
  uint32_t *kb = reinterpret_cast<uint32_t *>(smem);
  // comp[slot][i]: M of decoder sig[i] at the slot's column, then rewritten
  // in place into the queue-ordered prefix maximum of A (clamped at -1).
  // Rows are D + 1 words apart so that one row's writes to several slots fall
  // on different banks.
  const int Dp = D + 1;
  uint32_t *comp = kb + a.comp_off;
  int32_t *s_capq = reinterpret_cast<int32_t *>(kb + a.region);
  int32_t *s_sig = s_capq + D;
  int32_t *s_rank = s_sig + D;
  uint32_t *s_carry = reinterpret_cast<uint32_t *>(s_rank + D);
  int32_t *s_slot = reinterpret_cast<int32_t *>(s_carry + D);  // [W2] column -> slot (-1 none)
  int32_t *s_argA = s_slot + W2;                               // [W2]
  long long *s_maxA = reinterpret_cast<long long *>(
      (reinterpret_cast<uintptr_t>(s_argA + W2) + 15) & ~uintptr_t(15));  // [W2]
  uint64_t *s_bar = reinterpret_cast<uint64_t *>(s_maxA + W2);
  long long *s_segA = reinterpret_cast<long long *>(s_bar + 1);      // [8][32]
  int32_t *s_segrun = reinterpret_cast<int32_t *>(s_segA + kWarpsM * 32);  // [8][32]
  int32_t *s_segK = s_segrun + kWarpsM * 32;                          // [8][32]
  int32_t *s_need = s_segK + kWarpsM * 32;                            // [W2] column needs PMq
  int32_t *s_needlist = s_need + W2;                                  // [W2]
  __shared__ int s_nslots, s_abort, s_nneed;

  const Unit un = a.units[unit];
  const int64_t t0 = static_cast<int64_t>(un.tile) * W2;
  if (tid == 0) {
    s_abort = 0;
    if (a.use_tma) {
      mbar_init(s_bar, 1);
      fence_mbar_init();
      // every box is credited in full, rows past D included (zero-filled)
      mbar_expect_tx(s_bar, static_cast<uint32_t>(a.boxes) * a.box_rows * W2 * 4u);
      for (int b = 0; b < a.boxes; ++b)
        tma_load_2d(kb + static_cast<size_t>(b) * a.box_rows * W2, &tmap, s_bar, un.tile * W2,
                    b * a.box_rows);
    }
  }
  // queue order, capacities and this tile's carries; columns this unit needs
  for (int k = tid; k < D; k += kMainThreads) {
    s_sig[k] = __ldg(a.sig + k);
    s_rank[k] = __ldg(a.rank_of + k);
    s_capq[k] = __ldg(a.capq + k);
    s_carry[k] = __ldg(a.carry + static_cast<int64_t>(k) * a.T2 + un.tile);
  }
  for (int c = tid; c < W2; c += kMainThreads) s_slot[c] = 0;
  __syncthreads();
  for (int q0 = 0; q0 < un.count; q0 += kMainThreads * 8) {
    int32_t uu[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {  // issue the loads together
      const int q = q0 + i * kMainThreads + tid;
      uu[i] = q < un.count ? __ldg(a.su + un.start + q) : 0;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (uu[i] > 0) s_slot[uu[i] - 1 - t0] = 1;
  }
  if (!a.use_tma) {
    for (int e = tid; e < D * W2; e += kMainThreads) {
      const int r = e / W2, c = e - (e / W2) * W2;
      const int64_t t = t0 + c;
      // 32-column tiles use the layout of a 128-byte swizzled TMA copy
      const int at = W2 == 32 ? r * 32 + ((((c >> 2) ^ (r & 7))) << 2) + (c & 3) : e;
      kb[at] = t < H ? static_cast<uint32_t>(a.K[static_cast<int64_t>(r) * H + t]) : 0u;
    }
  }
  __syncthreads();
  if (warp == 0) {  // compact the flagged columns (W2 <= 256)
    int run = 0;
    for (int c0 = 0; c0 < W2; c0 += 32) {
      const int c = c0 + lane;
      const bool f = c < W2 && s_slot[c] != 0;
      const unsigned bal = __ballot_sync(0xffffffffu, f);
      if (c < W2) s_slot[c] = f ? run + __popc(bal & lanemask_lt()) : -1;
      run += __popc(bal);
    }
    if (lane == 0) s_nslots = run;
  }
  if (a.use_tma && !mbar_wait_bounded(s_bar, 0)) {
    if (tid == 0) flag_error(a.status, MAPS_E_TIMEOUT);
    s_abort = 1;
  }
  __syncthreads();
  if (s_abort) {
    // a copy may still land: wait for it once more (bounded) before leaving
    mbar_wait_bounded(s_bar, 0);
    return;
  }
  const int nslots = s_nslots;

  // --- prefix maximum of K + t along each row; keep the needed columns ----
  bool neg = false;
  if (W2 == 32 && a.alias) {
    // One row per thread (D <= kMainThreads): every row is read into registers
    // first, then, after a barrier, comp is written over the tile.
    const int row = tid;
    const bool live = row < D;
    uint4 q[8];
    if (live) {
      const uint4 *rp = reinterpret_cast<const uint4 *>(kb + static_cast<size_t>(row) * 32);
#pragma unroll
      for (int ch = 0; ch < 8; ++ch) q[ch] = rp[ch ^ (row & 7)];
    }
    __syncthreads();  // the tile has been read: its space becomes comp
    if (live) {
      uint32_t run = s_carry[row];
      const int rk = s_rank[row];
#pragma unroll
      for (int ch = 0; ch < 8; ++ch) {
        const uint32_t raw[4] = {q[ch].x, q[ch].y, q[ch].z, q[ch].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int c = ch * 4 + e;
          const int64_t t = t0 + c;
          if (t < H) {
            if (static_cast<int32_t>(raw[e]) < 0) neg = true;
            const uint32_t x = raw[e] + static_cast<uint32_t>(t);  // K + t < 2^32
            run = x > run ? x : run;
          }
          const int sl = s_slot[c];
          if (sl >= 0) comp[static_cast<size_t>(sl) * Dp + rk] = run;
        }
      }
    }
  } else if constexpr (W2 == 32) {
    // One thread per row.  The tile is stored with 128-byte swizzling: the
    // 16-byte chunk ch of row r sits at chunk ch ^ (r & 7) of its 128-byte
    // row, so a warp loading one chunk of 32 rows hits every bank once per
    // quarter-warp.  The running maximum starts from the row's carry.
    for (int row = tid; row < D; row += kMainThreads) {
      const uint4 *rp = reinterpret_cast<const uint4 *>(kb + static_cast<size_t>(row) * 32);
      uint32_t run = s_carry[row];
      const int rk = s_rank[row];
#pragma unroll
      for (int ch = 0; ch < 8; ++ch) {
        const uint4 q = rp[ch ^ (row & 7)];
        const uint32_t raw[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int c = ch * 4 + e;
          const int64_t t = t0 + c;
          if (t < H) {
            if (static_cast<int32_t>(raw[e]) < 0) neg = true;
            const uint32_t x = raw[e] + static_cast<uint32_t>(t);  // K + t < 2^32
            run = x > run ? x : run;
          }
          const int sl = s_slot[c];
          if (sl >= 0) comp[static_cast<size_t>(sl) * Dp + rk] = run;
        }
      }
    }
  } else {
    constexpr int seg = W2 / 16;  // cells per row segment; 16 segments per row
    const int items = ((D * 16 + kMainThreads - 1) / kMainThreads) * kMainThreads;
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
        const uint32_t cr = s_carry[row];
        const int rk = s_rank[row];
        excl = excl > cr ? excl : cr;
#pragma unroll
        for (int j = 0; j < seg; ++j) {
          const int sl = s_slot[sg * seg + j];
          if (sl >= 0) comp[static_cast<size_t>(sl) * Dp + rk] = v[j] > excl ? v[j] : excl;
        }
      }
    }
  }
  if (neg) flag_error(a.status, MAPS_E_RANGE);
  __syncthreads();

  // --- per needed column: arg-max of A, then (where some candidate can be
  // placed) the prefix maximum of A in queue order ---------------------------
  // Columns go 32 at a time, lane c taking column cb + c; warp w takes the
  // w-th eighth of the queue positions, in order.  Rows are D + 1 words apart,
  // so a warp's 32 columns fall on 32 banks.
  {
    const int L = (D + kWarpsM - 1) / kWarpsM;
    const int i0 = warp * L, i1 = min(D, i0 + L);
    // (1) the best (A, decoder) of each column: each segment's, then warp 0
    // combines the eight
    for (int cb = 0; cb < nslots; cb += 32) {
      const int sl = cb + lane;
      const bool live = sl < nslots;
      const uint32_t *col = comp + static_cast<size_t>(live ? sl : 0) * Dp;
      long long bA = LLONG_MIN;
      int bK = 0x7fffffff;
      if (live)
        for (int i = i0; i < i1; ++i) {
          const long long A = static_cast<long long>(s_capq[i]) - 1 - static_cast<long long>(col[i]);
          const int k = s_sig[i];
          if (A > bA || (A == bA && k < bK)) {
            bA = A;
            bK = k;
          }
        }
      s_segA[warp * 32 + lane] = bA;
      s_segK[warp * 32 + lane] = bK;
      __syncthreads();
      if (live && warp == 0) {
        for (int w = 1; w < kWarpsM; ++w) {
          const long long yA = s_segA[w * 32 + lane];
          const int yK = s_segK[w * 32 + lane];
          if (yA > bA || (yA == bA && yK < bK)) {
            bA = yA;
            bK = yK;
          }
        }
        s_maxA[sl] = bA;
        s_argA[sl] = bK;
        s_need[sl] = 0;
      }
      __syncthreads();  // the segment arrays serve the next 32 columns
    }
    // (2) a candidate that fits no decoder (p above its column's best A) is
    // decided here (most headroom); the others mark their column
    for (int q = tid; q < un.count; q += kMainThreads) {
      const int32_t p = __ldg(a.sp + un.start + q);
      const int sl = s_slot[__ldg(a.su + un.start + q) - 1 - t0];
      if (static_cast<long long>(p) <= s_maxA[sl]) {
        s_need[sl] = 1;
      } else {
        const int j = __ldg(a.ord + un.start + q);
        a.choice[j] = s_argA[sl];
        if (a.headroom) a.headroom[j] = s_maxA[sl] - p;
      }
    }
    __syncthreads();
    if (warp == 0) {  // compact them
      int run = 0;
      for (int c0 = 0; c0 < nslots; c0 += 32) {
        const int sl = c0 + lane;
        const bool f = sl < nslots && s_need[sl] != 0;
        const unsigned bal = __ballot_sync(0xffffffffu, f);
        if (f) s_needlist[run + __popc(bal & lanemask_lt())] = sl;
        run += __popc(bal);
      }
      if (lane == 0) s_nneed = run;
    }
    __syncthreads();
    // (3) for those: a running maximum of A (clamped at -1) per segment,
    // written in place, then each segment raised to the maximum of the
    // segments before it
    const int nneed = s_nneed;
    for (int cb = 0; cb < nneed; cb += 32) {
      const bool live = cb + lane < nneed;
      const int sl = live ? s_needlist[cb + lane] : 0;
      uint32_t *col = comp + static_cast<size_t>(sl) * Dp;
      int32_t run = -1;
      if (live)
        for (int i = i0; i < i1; ++i) {
          const long long A = static_cast<long long>(s_capq[i]) - 1 - static_cast<long long>(col[i]);
          const int32_t a32 = A < -1 ? -1 : static_cast<int32_t>(A);
          run = a32 > run ? a32 : run;
          col[i] = static_cast<uint32_t>(run);
        }
      s_segrun[warp * 32 + lane] = run;
      __syncthreads();
      if (live) {
        int32_t ex = -1;
        for (int w = 0; w < warp; ++w) ex = max(ex, s_segrun[w * 32 + lane]);
        if (ex > -1)
          for (int i = i0; i < i1; ++i) {
            const int32_t v = static_cast<int32_t>(col[i]);
            if (v < ex) col[i] = static_cast<uint32_t>(ex);
          }
      }
      __syncthreads();
    }
  }

  // --- the candidates that fit some decoder (loads issued together, then the
  // searches); the others were decided above ----------------------------------
  for (int q0 = 0; s_nneed > 0 && q0 < un.count; q0 += kMainThreads * 8) {
    int32_t pp[8], uu[8], jj[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int q = q0 + i * kMainThreads + tid;
      const bool ok = q < un.count;
      pp[i] = ok ? __ldg(a.sp + un.start + q) : 0;
      uu[i] = ok ? __ldg(a.su + un.start + q) : 0;
      jj[i] = ok ? __ldg(a.ord + un.start + q) : -1;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      if (jj[i] < 0) continue;
      const int32_t p = pp[i];
      const int c = static_cast<int>(uu[i] - 1 - t0);
      const int sl = s_slot[c];
      if (s_maxA[sl] < p) continue;  // nothing feasible: decided above
      const int32_t *pm = reinterpret_cast<const int32_t *>(comp) + static_cast<size_t>(sl) * Dp;
      int l = 0, r = D - 1;  // first queue position whose prefix reaches p
      while (l < r) {
        const int mid = (l + r) >> 1;
        if (pm[mid] >= p)
          r = mid;
        else
          l = mid + 1;
      }
      a.choice[jj[i]] = s_sig[l];
      if (a.headroom) a.headroom[jj[i]] = static_cast<long long>(pm[l]) - p;
    }
  }
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
// mc: rank every decoder by headroom alone (the memory-only ablation): all
// picks take the infeasible class, whose order is the largest headroom first.
__device__ __forceinline__ Pick make_pick(long long h, int32_t q, int k, bool mc = false) {
  Pick p;
  const bool feas = h >= 0 && !mc;
  p.inf = feas ? 0 : 1;
  p.v = feas ? static_cast<long long>(q) : -h;
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
// SEQUENTIAL horizon dispatch: one block walks the candidates in order.
// Scoring decoder k needs M_k(u) = max_{t<u} (K[k][t] + t); it is read from
// the 16-step summary kmax (built from K just before) for the whole blocks
// below u plus at most 15 cells of K.  Reserving the footprint adds
// p + t + 1 to K[k*][t] for t < u and rebuilds the summary entries of the
// blocks it touched, so the summary always matches K.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024, 1)
dispatch_sequential_kernel(int D, int H, int32_t *K, uint32_t *kmax, const int32_t *cap,
                           int32_t *Q, int64_t J, const int32_t *cp, const int32_t *cb,
                           int32_t *choice, int64_t *headroom, int mc, int32_t *status) {
  pdl_prologue();
  __shared__ uint32_t s_M[kMaxD];
  __shared__ Pick s_w[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const int64_t nb = (static_cast<int64_t>(H) + kSumBlock - 1) / kSumBlock;
  bool bad = false;
  for (int k = tid; k < D; k += blockDim.x)
    if ((cap[k] | Q[k]) < 0) bad = true;
  if (bad) flag_error(status, MAPS_E_RANGE);  // K < 0 is reported by the summary pass
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
    const int nfull = u / kSumBlock, rem = u - nfull * kSumBlock;
    for (int k = warp; k < D; k += nwarp) {
      const uint32_t *km = kmax + static_cast<int64_t>(k) * nb;
      const int32_t *row = K + static_cast<int64_t>(k) * H;
      uint32_t m = 0;
      for (int b = lane; b < nfull; b += 32) m = max(m, km[b]);
      if (lane < rem) {
        const int t = nfull * kSumBlock + lane;
        m = max(m, static_cast<uint32_t>(row[t]) + static_cast<uint32_t>(t));
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, off));
      if (lane == 0) s_M[k] = m;
    }
    __syncthreads();
    Pick mine = no_pick();
    for (int k = tid; k < D; k += blockDim.x) {
      const long long h = static_cast<long long>(cap[k]) - (static_cast<long long>(p) + 1 + s_M[k]);
      const Pick c = make_pick(h, Q[k], k, mc != 0);
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
    // reserve the candidate's footprint at the chosen decoder; the blocks it
    // touches are whole 16-lane groups of the loop, so a group's shuffle
    // maximum is that block's new summary entry
    int32_t *row = K + static_cast<int64_t>(b.k) * H;
    uint32_t *km = kmax + static_cast<int64_t>(b.k) * nb;
    const int end = min(((u + kSumBlock - 1) / kSumBlock) * kSumBlock, H);
    bool over = false;
    for (int t0 = 0; t0 < end; t0 += blockDim.x) {
      const int t = t0 + tid;
      uint32_t x = 0;
      if (t < end) {
        long long v = row[t];
        if (t < u) {
          v += static_cast<long long>(p) + t + 1;
          if (v > 0x7fffffffLL) {
            over = true;
            v = 0x7fffffffLL;
          }
          row[t] = static_cast<int32_t>(v);
        }
        x = static_cast<uint32_t>(v) + static_cast<uint32_t>(t);
      }
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) x = max(x, __shfl_xor_sync(0xffffffffu, x, off));
      if ((lane & (kSumBlock - 1)) == 0 && t < end) km[t / kSumBlock] = x;
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
  pdl_prologue();
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
  pdl_prologue();
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
  pdl_prologue();
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
  int box_rows, boxes, Drows, W2, T2, tile_stride, comp_off, region;
  bool alias;
  size_t smem;
};

SnapGeom snap_geom(int D, int H) {
  SnapGeom g;
  g.box_rows = D < kBoxRows ? D : kBoxRows;
  g.boxes = (D + g.box_rows - 1) / g.box_rows;
  g.Drows = g.boxes * g.box_rows;
  int w = 256;
  while (w > 16 && static_cast<long long>(w) * g.Drows > 8192) w >>= 1;
  g.W2 = w;
  g.T2 = static_cast<int>((static_cast<long long>(H) + w - 1) / w);
  g.tile_stride = (g.Drows * w + 255) / 256 * 256;  // 1 KB-aligned buffer
  // with 32-column tiles and at most one row per thread, comp (the prefix
  // maxima, padded rows) overwrites the tile once every row is in registers
  const int comp_words = (D + 1) * w;
  g.alias = w == 32 && D <= kMainThreads;
  g.comp_off = g.alias ? 0 : g.tile_stride;
  g.region = g.alias ? std::max(g.tile_stride, comp_words) : g.tile_stride + comp_words;
  size_t b = static_cast<size_t>(g.region) * 4;       // K tile and comp
  b += 4 * static_cast<size_t>(D) * 4;                // capq, sig, rank, carry
  b += 2 * static_cast<size_t>(w) * 4;                // slot, argA
  b += 16;                                            // alignment slack
  b += static_cast<size_t>(w) * 8;                    // maxA
  b += 8;                                             // barrier
  b += static_cast<size_t>(kMainThreads) * (8 + 4 + 4);  // per-segment partials [8][32]
  b += 2 * static_cast<size_t>(w) * 4;                    // columns needing PMq, their list
  g.smem = b;
  return g;
}

struct SnapWs {
  uint32_t *zero;  // tcount[T2], tcursor[T2], nunits, ticket (zeroed per call)
  size_t zero_words;
  uint32_t *toff;
  Unit *units;
  int32_t *ord, *sp, *su;
  int32_t *sig, *rank_of, *capq;
  uint32_t *carry;  // [D][T2]
  uint32_t *kmax;   // [D][ceil(H/16)], used when the caller passes none
  int64_t max_units;
};

SnapWs carve_snap(Carve &c, int D, int H, int T2, int64_t J) {
  SnapWs w;
  w.zero_words = 2 * static_cast<size_t>(T2) + 2;  // tcount, tcursor, nunits, ticket
  w.zero = c.take<uint32_t>(w.zero_words);
  w.toff = c.take<uint32_t>(static_cast<size_t>(T2) + 1);
  w.max_units = static_cast<int64_t>(T2) + (J + kUnitCands - 1) / kUnitCands;
  w.units = c.take<Unit>(static_cast<size_t>(w.max_units) + 1);
  const size_t nj = static_cast<size_t>(J > 0 ? J : 1);
  w.ord = c.take<int32_t>(nj);
  w.sp = c.take<int32_t>(nj);
  w.su = c.take<int32_t>(nj);
  w.sig = c.take<int32_t>(static_cast<size_t>(D));
  w.rank_of = c.take<int32_t>(static_cast<size_t>(D));
  w.capq = c.take<int32_t>(static_cast<size_t>(D));
  w.carry = c.take<uint32_t>(static_cast<size_t>(T2) * D);
  w.kmax = c.take<uint32_t>(static_cast<size_t>(D) * ((static_cast<size_t>(H) + kSumBlock - 1) / kSumBlock));
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

// Events recorded around the scoring kernel (maps_set_dispatch_events).
thread_local cudaEvent_t g_score_ev[2] = {nullptr, nullptr};

template <int W2>
int run_snapshot(int64_t grid, size_t smem, cudaStream_t s, const CUtensorMap &tmap, const SnapArgs &a) {
  MAPS_TRY(cuda_ok(cudaFuncSetAttribute(dispatch_snapshot_kernel<W2>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(smem))));
  if (g_score_ev[0]) MAPS_TRY(cuda_ok(cudaEventRecord(g_score_ev[0], s)));
  launch_pdl(dispatch_snapshot_kernel<W2>, static_cast<unsigned>(grid), kMainThreads, smem, s, tmap, a);
  MAPS_TRY(launch_ok());
  if (g_score_ev[1]) MAPS_TRY(cuda_ok(cudaEventRecord(g_score_ev[1], s)));
  return MAPS_OK;
}

int launch_snapshot(int D, int H, const int32_t *K, const uint32_t *kmax, const int32_t *cap,
                    const int32_t *Q, int64_t J, const int32_t *cp, const int32_t *cb,
                    int32_t *choice, int64_t *headroom, void *ws, cudaStream_t s) {
  const SnapGeom g = snap_geom(D, H);
  if (g.smem + 1024 > static_cast<size_t>(max_smem_optin())) return MAPS_E_INVALID;
  Carve cv(ws);
  const SnapWs w = carve_snap(cv, D, H, g.T2, J);
  if (w.max_units > 0x7fffffffLL) return MAPS_E_INVALID;
  int32_t *status = status_word(ws);
  uint32_t *tcount = w.zero, *tcursor = w.zero + g.T2;
  uint32_t *nunits = w.zero + 2 * static_cast<size_t>(g.T2);
  uint32_t *ticket = nunits + 1;  // bin_count blocks finished
  const int sms = sm_count();
  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.zero, 0, w.zero_words * 4, s)));
  const bool check_kmax = kmax != nullptr;
  if (kmax == nullptr) {
    const int64_t nb = (static_cast<int64_t>(H) + kSumBlock - 1) / kSumBlock;
    const int gk = static_cast<int>(std::min<int64_t>((nb * D + 255) / 256, 8LL * sms));
    launch_pdl(kmax_from_K_kernel, gk, 256, 0, s, D, H, K, w.kmax, status);
    kmax = w.kmax;
  }
  // carries of D decoders, and candidate counts in blocks of 256 candidates
  const int gc = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((J + 255) / 256, 4LL * sms)));
  launch_pdl(dispatch_prep_kernel, D + gc, 256, 0, s, D, D, H, g.W2, g.T2, K, check_kmax, kmax,
             w.carry, Q, cap,
             w.sig, w.rank_of, w.capq, J, cp, cb, tcount, choice, headroom, status, ticket, w.toff,
             w.units, nunits);
  const int gb = static_cast<int>(std::min<int64_t>((J + 255) / 256, 4LL * sms));
  launch_pdl(bin_scatter_kernel, gb, 256, 0, s, J, H, g.W2, g.T2, cp, cb, w.toff, tcursor, w.ord,
             w.sp, w.su);
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
                           g.W2 == 32 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
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
  a.comp_off = g.comp_off;
  a.region = g.region;
  a.alias = g.alias;
  a.use_tma = use_tma;
  a.K = K;
  a.sig = w.sig;
  a.rank_of = w.rank_of;
  a.capq = w.capq;
  a.carry = w.carry;
  a.units = w.units;
  a.nunits = nunits;
  a.ord = w.ord;
  a.sp = w.sp;
  a.su = w.su;
  a.choice = choice;
  a.headroom = headroom;
  a.status = status;
  const int64_t grid = std::max<int64_t>(1, w.max_units);  // units past *nunits return at once
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

namespace maps {
int dispatch_sequential(int D, int H, int32_t *K, const int32_t *cap, int32_t *Q, int64_t J,
                        const int32_t *cp, const int32_t *cb, int32_t *choice, int64_t *headroom,
                        bool mc, void *ws, cudaStream_t s) {
  // a private summary of K (also validating K >= 0); updated in place
  int32_t *status = status_word(ws);
  Carve cv(ws);
  const int64_t nb = (static_cast<int64_t>(H) + kSumBlock - 1) / kSumBlock;
  uint32_t *km = cv.take<uint32_t>(static_cast<size_t>(D) * nb);
  const int gk = static_cast<int>(std::min<int64_t>((nb * D + 255) / 256, 8LL * sm_count()));
  launch_pdl(kmax_from_K_kernel, gk, 256, 0, s, D, H, K, km, status);
  launch_pdl(dispatch_sequential_kernel, 1, 1024, 0, s, D, H, K, km, cap, Q, J, cp, cb, choice,
             headroom, mc ? 1 : 0, status);
  return launch_ok();
}
}  // namespace maps

extern "C" {

int maps_set_dispatch_events(void *before, void *after) {
  maps::g_score_ev[0] = static_cast<cudaEvent_t>(before);
  maps::g_score_ev[1] = static_cast<cudaEvent_t>(after);
  return MAPS_OK;
}

size_t maps_dispatch_workspace_size(int32_t mode, int32_t D, int32_t H, int64_t J) {
  using namespace maps;
  Carve c(nullptr);
  if (mode == MAPS_MODE_SNAPSHOT && D >= 1 && H >= 1 && H <= kMaxH) {
    const SnapGeom g = snap_geom(D, H);
    carve_snap(c, D, H, g.T2, J);
  } else if (mode == MAPS_MODE_SEQUENTIAL && D >= 1 && H >= 1 && H <= kMaxH) {
    c.take<uint32_t>(static_cast<size_t>(D) * ((static_cast<size_t>(H) + kSumBlock - 1) / kSumBlock));
  } else if ((mode == MAPS_MODE_ALG1_SNAPSHOT || mode == MAPS_MODE_ALG1_SEQUENTIAL) && D >= 1) {
    c.take<long long>(static_cast<size_t>(D));
  }
  return c.bytes();
}

int maps_dispatch(int32_t mode, int32_t D, int32_t H, int32_t S, int32_t *K, const uint32_t *kmax,
                  const int32_t *cap, int32_t *Q, const int64_t *res_off, int64_t R, const int32_t *prompt,
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
      return launch_snapshot(D, H, K, kmax, cap, Q, J, cand_prompt, cand_bound, choice_out,
                             headroom_out, ws, s);
    case MAPS_MODE_SEQUENTIAL:
      return dispatch_sequential(D, H, K, cap, Q, J, cand_prompt, cand_bound, choice_out,
                                 headroom_out, false, ws, s);
    default: {
      Carve cv(ws);
      long long *B_eff = cv.take<long long>(static_cast<size_t>(D));
      launch_pdl(alg1_budget_kernel, D, 256, 0, s, D, S, res_off, R, prompt, gen, bound, cap, B_eff, status);
      if (mode == MAPS_MODE_ALG1_SNAPSHOT) {
        const int grid = static_cast<int>(std::min<int64_t>((J + 255) / 256, 4LL * sm_count()));
        launch_pdl(alg1_snapshot_kernel, grid, 256, 0, s, D, S, B_eff, cap, Q, J, cand_prompt, cand_bound,
                                                  choice_out, headroom_out, status);
      } else {
        launch_pdl(alg1_sequential_kernel, 1, 1024, 0, s, D, S, B_eff, cap, Q, J, cand_prompt, cand_bound,
                                                  choice_out, headroom_out, status);
      }
      return launch_ok();
    }
  }
}

}  // extern "C"
