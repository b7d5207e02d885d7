// order.cu -- local SJF reordering with max-wait promotion (Sec. 3.3).
//
// The queue order is the lexicographic order of
//     (decoder, not promoted, promoted ? arrival : bound, arrival, index).
// It is computed as a stable least-significant-digit radix sort of 8-bit
// digits over a compact key:
//   * entries are first put in arrival order (stable), unless arrival is
//     already non-decreasing in index, which the first pass checks;
//   * the key is then  decoder << (1 + ub) | not_promoted << ub | (not
//     promoted ? bound : 0), with ub the bit width of the largest bound of a
//     non-promoted entry: promoted entries need no primary key because the
//     arrival order is already in place and the sort is stable;
//   * a key of at most 32 bits is sorted as 32 bits, otherwise as 64 bits.
// Small calls (at most kSegMax entries and kSmallOrderD decoders) take one
// block, order_small_kernel, with the whole order in shared memory.
// Otherwise the kernels are a prep pass (validation, largest bound, entries
// per decoder, arrival order check; its last block chooses the form), a key
// pass, the segment sort, and a cooperative finishing kernel.
// Segmented form (arrival non-decreasing along the index): the key pass
// scatters each entry's index to its decoder's segment; one block sorts a
// segment of at most kSegMax entries in shared memory on (not promoted,
// primary, index), a unique key, and a longer segment is sorted as chunks of
// kSegMax whose runs the finishing kernel ranks pairwise (up to kPairRuns
// chunks) or merges pairwise level by level.
// Otherwise the finishing kernel plans and runs one global sweep per digit:
// tiles of 4096 keys are ranked stably in shared memory, each tile learns its
// offsets from earlier tiles by decoupled look-back (one thread per digit
// walks back over packed flag-and-count words until it meets an inclusive
// prefix), and writes out bin by bin.  Kernels of the form not taken return
// at once, so the host never waits on the device.
#include "maps_internal.cuh"
#include "maps_bench.h"

#include <algorithm>


namespace maps {
namespace {

constexpr int kRadix = 256;
constexpr int kPassThreads = 512;
constexpr int kIPT = 8;
constexpr int kTile = kPassThreads * kIPT;  // 4096 keys per tile
constexpr int kPassWarps = kPassThreads / 32;
constexpr int kLoPasses = 4;  // arrival digits
constexpr int kHiPasses = 8;  // key digits
constexpr int kPasses = kLoPasses + kHiPasses;
constexpr int kDecSmem = 8192;  // decoders counted in shared memory up to this D
constexpr uint32_t kFlagAgg = 1, kFlagInc = 2;

enum : int32_t { kBufA = 0, kBufB = 1, kHiIdentity = 2, kPermOut = 2 };

// Test aid (maps_test_withhold_lookback): a tile of the global form's passes
// that publishes nothing to the look-back (-1: none), and the polls a
// look-back wait makes before it gives up.
__device__ int32_t g_withheld_tile = -1;
__device__ uint32_t g_lookback_spins = kSpinLimit;
// Test aid (maps_test_absent_block): a block of the finishing kernel that
// returns at once, so that the others' grid barrier runs out (-1: none).  The
// barrier waits also give up after g_lookback_spins polls.
__device__ int32_t g_absent_block = -1;

struct OrderCounts {
  uint32_t h[kPasses][kRadix];
  uint32_t unsorted;   // arrival decreases somewhere along the index
  uint32_t max_bound;  // largest bound of a non-promoted entry
  uint32_t segmented;  // decoder segments are sorted in shared memory
  uint32_t nitems;     // segments and chunks to sort
  uint32_t nmtiles;    // merge tiles of the long queues
  uint32_t max_levels; // merge levels the longest queue needs
  uint32_t done_blocks;  // prep blocks finished
  uint32_t stable;     // segmented form with the decoder scatter in index order
  uint32_t npairs;     // run pairs reserved by the pairwise-ranked long queues
  uint32_t npairq;     // pairwise-ranked long queues
};

// Segmented form: when arrival is non-decreasing along the index (so arrival
// order is index order) and every decoder's queue fits in shared memory, the
// entries are scattered to their decoder's segment in any order and each
// segment is sorted by one block on the key (not promoted, primary, index),
// which is unique, so no pass has to be stable across blocks.
// With at most kStableD decoders the scatter keeps index order within each
// decoder (stable): the prep and key passes split the entries into the same
// contiguous block ranges, the prep pass counts each block's entries per
// decoder, its last block turns the counts into each block's first slot in
// every segment, and the key pass ranks the entries of a round in index order.
// The segment sort then needs no index digits.
constexpr int kStableD = 1024;
constexpr int kPrepBlocks = 304;    // prep and key blocks at most
constexpr int kGroupBlocks = 16;    // prep blocks whose counts are also summed per group
constexpr int kKeysU = 4;           // entries per thread per round
constexpr int kKeysRound = 512 * kKeysU;
__host__ __device__ __forceinline__ int64_t prep_chunk(int64_t N) {
  const int64_t per = (N + kPrepBlocks - 1) / kPrepBlocks;
  const int64_t c = (per + kKeysRound - 1) / kKeysRound * kKeysRound;
  return c > kKeysRound ? c : kKeysRound;
}
// The bucketed form (order_bucket_kernel): entries per thread per round, and
// its blocks' ranges (whole rounds, at most kPrepBlocks blocks).
constexpr int kBucketU = 8;
constexpr int kBucketRound = 512 * kBucketU;
__host__ __device__ __forceinline__ int64_t bucket_chunk(int64_t N) {
  const int64_t per = (N + kPrepBlocks - 1) / kPrepBlocks;
  const int64_t c = (per + kBucketRound - 1) / kBucketRound * kBucketRound;
  return c > kBucketRound ? c : kBucketRound;
}
constexpr int kSegThreads = 512;
constexpr int kSegIPT = 9;
constexpr int kSegMax = kSegThreads * kSegIPT;  // entries one block sorts
// A longer queue is sorted as chunks of kSegMax entries, whose sorted runs are
// then merged pairwise, level by level, in tiles of kMergeTile outputs
// (kMergeTile divides kSegMax, so no tile straddles two runs).
constexpr int kMergeTile = 512;
constexpr int kMergeThreads = 512;  // the finishing kernel's block
static_assert(kSegMax % kMergeTile == 0, "merge tiles align with runs");

// A long queue of at most kPairRuns chunks is ranked pairwise instead: for
// every ordered pair of its sorted runs (A, B) one block counts, for each key
// of A, the keys of B below it (the keys are unique); after one grid barrier
// a key's place in the queue is its place in A plus those counts.  The counts
// are 16-bit, [pair][position in A]; the pairs a call may use are capped by
// pair_budget(N), and a queue past the cap or past kPairRuns is merged.
constexpr int kPairRuns = 16;
__host__ __device__ __forceinline__ int64_t pair_budget(int64_t N) {
  // room for one queue of every entry (up to kPairRuns runs), and at larger
  // N four pairs per chunk
  const int64_t runs = (N + kSegMax - 1) / kSegMax;
  const int64_t r = runs < kPairRuns ? runs : kPairRuns;
  const int64_t per = 4 * (N / kSegMax);
  const int64_t b = per > r * (r - 1) ? per : r * (r - 1);
  return b < 1024 ? b : 1024;
}
struct PairQueues {
  int64_t *off;    // [queue] first slot of the queue
  int32_t *n;      // [queue] entries
  int32_t *pair0;  // [queue] first pair id
  uint16_t *cnt;   // [pair][kSegMax] keys of B below each key of A
  int64_t budget;  // pairs the workspace holds
};

// Merge levels a queue of n entries needs: ceil(log2(ceil(n / kSegMax))).
__host__ __device__ __forceinline__ int merge_levels(int64_t n) {
  int64_t runs = (n + kSegMax - 1) / kSegMax;
  int l = 0;
  while ((int64_t(1) << l) < runs) ++l;
  return l;
}
constexpr int kSegWarps = kSegThreads / 32;
__device__ __forceinline__ int index_bits(int64_t N) {
  return N > 1 ? 64 - __clzll(static_cast<unsigned long long>(N - 1)) : 1;
}

struct OrderPlan {
  int32_t active[kPasses];
  int32_t src[kPasses];
  int32_t dst[kPasses];
  int32_t shift[kPasses];
  int32_t gather_buf;  // -1: none
  int32_t npasses;
  int32_t wide;        // keys need 64 bits
  int32_t ubits;       // bit width of the primary (bound) field
  int32_t ordinal[kPasses];  // position among the active passes
  uint32_t digit_off[kPasses][kRadix];
};

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Warp-aggregated shared-memory increment of bin `b` (all lanes present).
__device__ __forceinline__ void warp_count(uint32_t *hist, int b, bool valid) {
  const unsigned peers = __match_any_sync(0xffffffffu, valid ? b : -1);
  if (valid && static_cast<int>(threadIdx.x & 31) == __ffs(peers) - 1)
    atomicAdd(&hist[b], static_cast<uint32_t>(__popc(peers)));
}

__device__ __forceinline__ int bit_width(uint32_t x) { return x ? 32 - __clz(x) : 0; }

// Segmented form, step 1 (one block, run by the last prep block): decoder
// segment offsets, the sort items (a queue of at most kSegMax entries is one
// item whose sort writes the order; a longer one gives one item per chunk,
// marked by a negative count, whose sort writes keys for the merges) and the
// merge tiles of the long queues; the form applies when arrival is already
// in index order.
__device__ void seg_plan_block(int D, OrderCounts *counts, const uint32_t *dec_count,
                               int64_t *seg_off, int64_t *item_off, int32_t *item_n,
                               int32_t *item_dec, int64_t *mt_off, int32_t *mt_n, int32_t *mt_t,
                               PairQueues pq) {
  __shared__ long long s_w[32];
  __shared__ int s_bw[32];
  __shared__ long long s_carry;
  __shared__ int s_bcarry;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5, nt = blockDim.x;
  if (t == 0) {
    s_carry = 0;
    s_bcarry = 0;
  }
  __syncthreads();
  for (int base = 0; base <= D; base += nt) {
    const int k = base + t;
    const long long c = k < D ? __ldcg(dec_count + k) : 0;
    const int big = c > kSegMax ? 1 : 0;
    // sort items of decoder k: its queue, or its chunks; item indices follow
    // from a scan, in decoder order
    const int nch = big ? static_cast<int>((c + kSegMax - 1) / kSegMax) : 0;
    const int nit = c > 0 ? (big ? nch : 1) : 0;
    long long incl = c;
    int bincl = nit;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, off);
      const int by = __shfl_up_sync(0xffffffffu, bincl, off);
      if (lane >= off) {
        incl += y;
        bincl += by;
      }
    }
    if (lane == 31) {
      s_w[warp] = incl;
      s_bw[warp] = bincl;
    }
    __syncthreads();
    long long wb = 0;
    int bwb = 0;
    for (int w = 0; w < warp; ++w) {
      wb += s_w[w];
      bwb += s_bw[w];
    }
    const long long carry = s_carry;
    const int bcarry = s_bcarry;
    const long long start = carry + wb + incl - c;
    if (k <= D) seg_off[k] = start;
    const uint32_t it = static_cast<uint32_t>(bcarry + bwb + bincl - nit);
    if (k < D && c > 0 && !big) {
      item_off[it] = start;
      item_n[it] = static_cast<int32_t>(c);
      item_dec[it] = k;
    } else if (k < D && big) {
      for (int j = 0; j < nch; ++j) {
        item_dec[it + j] = k;
        item_off[it + j] = start + static_cast<int64_t>(j) * kSegMax;
        item_n[it + j] = -static_cast<int32_t>(min(static_cast<long long>(kSegMax), c - static_cast<long long>(j) * kSegMax));
      }
      bool paired = false;
      if (nch <= kPairRuns) {  // rank the runs pairwise when the budget allows
        const uint32_t np2 = static_cast<uint32_t>(nch * (nch - 1));
        const uint32_t p0 = atomicAdd(&counts->npairs, np2);
        if (static_cast<int64_t>(p0) + np2 <= pq.budget) {
          const uint32_t q = atomicAdd(&counts->npairq, 1u);
          pq.off[q] = start;
          pq.n[q] = static_cast<int32_t>(c);
          pq.pair0[q] = static_cast<int32_t>(p0);
          paired = true;
        }
      }
      if (!paired) {  // pairwise merges, level by level
        atomicMax(&counts->max_levels, static_cast<uint32_t>(merge_levels(c)));
        const int ntl = static_cast<int>((c + kMergeTile - 1) / kMergeTile);
        const uint32_t mt = atomicAdd(&counts->nmtiles, static_cast<uint32_t>(ntl));
        for (int j = 0; j < ntl; ++j) {
          mt_off[mt + j] = start;
          mt_n[mt + j] = static_cast<int32_t>(c);
          mt_t[mt + j] = j;
        }
      }
    }
    __syncthreads();
    if (t == nt - 1) {
      s_carry = carry + wb + incl;
      s_bcarry = bcarry + bwb + bincl;
    }
    __syncthreads();
  }
  const bool segmented = __ldcg(&counts->unsorted) == 0;
  const bool stable = segmented && D <= kStableD;
  if (t == 0) {
    counts->segmented = segmented ? 1u : 0u;
    counts->stable = stable ? 1u : 0u;
    counts->nitems = static_cast<uint32_t>(s_bcarry);
  }
}

// Pass 1: validation, largest non-promoted bound, entries per decoder, and
// whether arrival is non-decreasing.
__global__ void __launch_bounds__(512)
order_prep_kernel(int64_t N, int D, int64_t chunk, const int32_t *__restrict__ dec,
                  const int32_t *__restrict__ bound, const int32_t *__restrict__ wait,
                  const int32_t *__restrict__ arrival, int32_t max_wait, OrderCounts *counts,
                  uint32_t *dec_count, int32_t *status, int64_t *seg_off, int64_t *item_off,
                  int32_t *item_n, int32_t *item_dec, int64_t *mt_off, int32_t *mt_n, int32_t *mt_t,
                  PairQueues pq, uint32_t *blk, uint32_t *grp, int Dp) {
  pdl_prologue();
  __shared__ uint32_t s_dec[kDecSmem];
  __shared__ bool s_last;
  const bool dec_smem = D <= kDecSmem;
  if (dec_smem)
    for (int i = threadIdx.x; i < D; i += blockDim.x) s_dec[i] = 0;
  __syncthreads();
  bool bad = false, unsorted = false;
  uint32_t umax = 0;
  constexpr int kU = kKeysU;  // entries per thread per round, loads issued together
  // this block's contiguous range of entries (the key pass uses the same)
  const int64_t r_begin = static_cast<int64_t>(blockIdx.x) * chunk;
  const int64_t r_end = r_begin + chunk < N ? r_begin + chunk : N;
  for (int64_t i0 = r_begin; i0 < r_end; i0 += static_cast<int64_t>(blockDim.x) * kU) {
    int32_t d[kU], u[kU], w[kU], ar[kU], an[kU];
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + q * blockDim.x + threadIdx.x;
      const bool ok = i < r_end;
      d[q] = ok ? __ldg(dec + i) : -1;
      u[q] = ok ? __ldg(bound + i) : 0;
      w[q] = ok ? __ldg(wait + i) : 0;
      ar[q] = ok ? __ldg(arrival + i) : 0;
      an[q] = (ok && i + 1 < N) ? __ldg(arrival + i + 1) : 0x7fffffff;
    }
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + q * blockDim.x + threadIdx.x;
      int dd = -1;
      if (i < r_end) {
        dd = d[q];
        if (dd < 0 || dd >= D || u[q] < 0 || ar[q] < 0) {
          bad = true;
          dd = dd < 0 || dd >= D ? 0 : dd;
        }
        if (w[q] <= max_wait && u[q] > 0) umax = max(umax, static_cast<uint32_t>(u[q]));
        if (an[q] < ar[q]) unsorted = true;
      }
      // lanes of one decoder combine their count (residents come grouped by
      // decoder, so a warp is often a single decoder)
      const unsigned peers = __match_any_sync(0xffffffffu, dd);
      if (dd >= 0 && static_cast<int>(threadIdx.x & 31) == __ffs(peers) - 1)
        atomicAdd(dec_smem ? &s_dec[dd] : &dec_count[dd], static_cast<uint32_t>(__popc(peers)));
    }
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) umax = max(umax, __shfl_xor_sync(0xffffffffu, umax, off));
  if ((threadIdx.x & 31) == 0 && umax) atomicMax(&counts->max_bound, umax);
  if (__syncthreads_or(unsorted) && threadIdx.x == 0) atomicOr(&counts->unsorted, 1u);
  if (dec_smem) {
    if (D <= kStableD)  // this block's counts, and its group's, for the stable scatter
      for (int i = threadIdx.x; i < Dp; i += blockDim.x) {
        const uint32_t v = i < D ? s_dec[i] : 0u;
        blk[static_cast<int64_t>(blockIdx.x) * Dp + i] = v;
        if (v) atomicAdd(&grp[static_cast<int64_t>(blockIdx.x / kGroupBlocks) * Dp + i], v);
      }
    // blocks start their flush at different decoders so they do not collide
    const int rot = static_cast<int>((static_cast<int64_t>(blockIdx.x) * 97) % D);
    for (int i = threadIdx.x; i < D; i += blockDim.x) {
      const int k = (i + rot) % D;
      if (s_dec[k]) atomicAdd(&dec_count[k], s_dec[k]);
    }
  }
  // the last block to finish plans the segmented form
  // (one thread publishes the block's counts: the barrier orders every
  // thread's atomics before its fence, as a grid barrier does)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&counts->done_blocks, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    seg_plan_block(D, counts, dec_count, seg_off, item_off, item_n, item_dec, mt_off, mt_n, mt_t, pq);
  }
}

// Stable segmented form, first pass (D <= kStableD), in place of the prep
// and key passes: one read of the four inputs.  Block b takes the contiguous
// entries [b chunk, (b + 1) chunk) and
//   1. counts them per decoder: blk[b][d], added to the totals dec_count[d];
//   2. writes each entry's raw key (not promoted << 63 | primary << 32 |
//      index, the primary being the bound of a non-promoted entry, else 0)
//      to raw[b chunk + bst[b][d] + its rank among the block's entries of
//      decoder d in index order], bst[b][d] being the block's exclusive
//      prefix of its counts over the decoders: the block's entries bucketed
//      by decoder, stably;
//   3. validates, takes the largest non-promoted bound and checks that
//      arrival is non-decreasing along the index, as the prep pass does.
// The last block to finish plans the segments (seg_plan_block).  The segment
// sort then gathers decoder d's entries block by block, which is index order.
__global__ void __launch_bounds__(512, 2)
order_bucket_kernel(int64_t N, int D, int64_t chunk, int Dp, const int32_t *__restrict__ dec,
                    const int32_t *__restrict__ bound, const int32_t *__restrict__ wait,
                    const int32_t *__restrict__ arrival, int32_t max_wait, OrderCounts *counts,
                    uint32_t *dec_count, int32_t *status, int64_t *seg_off, int64_t *item_off,
                    int32_t *item_n, int32_t *item_dec, int64_t *mt_off, int32_t *mt_n,
                    int32_t *mt_t, PairQueues pq, uint32_t *blk, uint32_t *bst,
                    unsigned long long *raw) {
  pdl_prologue();
  extern __shared__ __align__(16) uint32_t bsm[];
  uint32_t *hw = bsm;                     // [kPassWarps][Dp] per-warp counts, then slot bases
  uint32_t *run = bsm + kPassWarps * Dp;  // [Dp] counts, then the next slot of each bucket
  __shared__ uint32_t s_w[kPassWarps];
  __shared__ bool s_last;
  constexpr int kU = kBucketU;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r_begin = static_cast<int64_t>(blockIdx.x) * chunk;
  const int64_t r_end = r_begin + chunk < N ? r_begin + chunk : N;
  // a range of one round keeps its loads in registers from the count to the
  // scatter (all of them issued together); longer ranges load twice
  const bool one = r_end - r_begin <= kBucketRound;
  // per entry only its decoder and raw key stay live: validation, the largest
  // bound and the arrival check are taken as the loads land
  int32_t d[kU];
  uint32_t kp[kU];  // not promoted << 31 | primary (the index follows from the position)
  bool bad = false, unsorted = false;
  uint32_t umax = 0;
  auto load = [&](int64_t i0, bool all) {
    int32_t u[kU], w[kU], ar[kU], an[kU], dr[kU];
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + warp * (32 * kU) + q * 32 + lane;
      const bool ok = i < r_end;
      dr[q] = ok ? __ldg(dec + i) : 0;
      // an entry of the range always has a decoder in [0, D): one out of the
      // domain is counted and placed at 0 (and flagged)
      d[q] = !ok ? -1 : (dr[q] < 0 || dr[q] >= D ? 0 : dr[q]);
      if (all) {
        u[q] = ok ? __ldg(bound + i) : 0;
        w[q] = ok ? __ldg(wait + i) : 0;
        ar[q] = ok ? __ldg(arrival + i) : 0;
        an[q] = (ok && i + 1 < N) ? __ldg(arrival + i + 1) : 0x7fffffff;
      }
    }
    if (!all) return;
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + warp * (32 * kU) + q * 32 + lane;
      if (i < r_end) {
        if (dr[q] < 0 || dr[q] >= D || u[q] < 0 || ar[q] < 0) bad = true;
        if (w[q] <= max_wait && u[q] > 0) umax = max(umax, static_cast<uint32_t>(u[q]));
        if (an[q] < ar[q]) unsorted = true;
      }
      const uint32_t np = w[q] > max_wait ? 0u : 1u;
      kp[q] = np ? (1u << 31) | static_cast<uint32_t>(u[q] < 0 ? 0 : u[q]) : 0u;
    }
  };
  for (int k = tid; k < Dp; k += blockDim.x) run[k] = 0;
  __syncthreads();
  // 1. counts
  for (int64_t i0 = r_begin; i0 < r_end; i0 += kBucketRound) {
    load(i0, one);
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const unsigned pe = __match_any_sync(0xffffffffu, d[q]);
      if (d[q] >= 0 && lane == __ffs(pe) - 1) atomicAdd(&run[d[q]], static_cast<uint32_t>(__popc(pe)));
    }
  }
  __syncthreads();
  {
    // block exclusive scan of the counts over the decoders (two per thread;
    // Dp <= 2 * blockDim.x), published with the counts
    const int k0 = 2 * tid;
    const uint32_t v0 = k0 < Dp ? run[k0] : 0u, v1 = k0 + 1 < Dp ? run[k0 + 1] : 0u;
    uint32_t incl = v0 + v1;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_w[warp] = incl;
    __syncthreads();
    uint32_t base = 0;
    for (int ww2 = 0; ww2 < warp; ++ww2) base += s_w[ww2];
    const uint32_t e0 = base + incl - v0 - v1;
    uint32_t *brow = blk + static_cast<int64_t>(blockIdx.x) * Dp;
    uint32_t *srow = bst + static_cast<int64_t>(blockIdx.x) * Dp;
    if (k0 < Dp) {
      brow[k0] = v0;
      srow[k0] = e0;
      run[k0] = e0;
      if (v0) atomicAdd(&dec_count[k0], v0);
    }
    if (k0 + 1 < Dp) {
      brow[k0 + 1] = v1;
      srow[k0 + 1] = e0 + v0;
      run[k0 + 1] = e0 + v0;
      if (v1) atomicAdd(&dec_count[k0 + 1], v1);
    }
  }
  __syncthreads();
  // 2. and 3., round by round in index order
  unsigned long long *out = raw + r_begin;
  for (int64_t i0 = r_begin; i0 < r_end; i0 += kBucketRound) {
    for (int k = tid; k < kPassWarps * Dp; k += blockDim.x) hw[k] = 0;
    if (!one) load(i0, true);
    __syncthreads();  // counts zeroed
    uint32_t rk[kU], base[kU];  // leader lane << 8 | rank in the group; group size, then base
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const unsigned pe = __match_any_sync(0xffffffffu, d[q]);
      const int leader = __ffs(pe) - 1;
      rk[q] = (static_cast<uint32_t>(leader) << 8) | static_cast<uint32_t>(__popc(pe & lanemask_lt()));
      base[q] = lane == leader ? static_cast<uint32_t>(__popc(pe)) : 0u;
    }
#pragma unroll
    for (int q = 0; q < kU; ++q)  // in item order, so ranks follow the index
      if (d[q] >= 0 && base[q] != 0) base[q] = atomicAdd(&hw[warp * Dp + d[q]], base[q]);
    __syncthreads();
    for (int k = tid; k < D; k += blockDim.x) {  // exclusive over the warps
      uint32_t r = run[k];
      for (int ww2 = 0; ww2 < kPassWarps; ++ww2) {
        const uint32_t c = hw[ww2 * Dp + k];
        hw[ww2 * Dp + k] = r;
        r += c;
      }
      run[k] = r;
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const uint32_t b = __shfl_sync(0xffffffffu, base[q], static_cast<int>(rk[q] >> 8));
      const int64_t i = i0 + warp * (32 * kU) + q * 32 + lane;
      if (d[q] >= 0)
        out[hw[warp * Dp + d[q]] + b + (rk[q] & 255u)] =
            (static_cast<unsigned long long>(kp[q]) << 32) | static_cast<unsigned long long>(i & 0xffffffff);
    }
    __syncthreads();  // the counts are zeroed again for the next round
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) umax = max(umax, __shfl_xor_sync(0xffffffffu, umax, off));
  if (lane == 0 && umax) atomicMax(&counts->max_bound, umax);
  if (__syncthreads_or(unsorted) && tid == 0) atomicOr(&counts->unsorted, 1u);
  // the last block to finish plans the segmented form (one thread publishes
  // the block's results: the barrier orders every thread's atomics before
  // its fence, as a grid barrier does)
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&counts->done_blocks, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    seg_plan_block(D, counts, dec_count, seg_off, item_off, item_n, item_dec, mt_off, mt_n, mt_t, pq);
  }
}

// The global form's key pass: each entry's key (decoder, not promoted,
// primary) in index order, its arrival digits where arrival is out of index
// order, and the histograms of every digit (sh: kPasses x kRadix words of
// shared memory).  Any grid; every thread of the block takes part.
__device__ void global_key_pass(int64_t N, int D, int dbits, const int32_t *__restrict__ dec,
                                const int32_t *__restrict__ bound, const int32_t *__restrict__ wait,
                                const int32_t *__restrict__ arrival, int32_t max_wait,
                                OrderCounts *counts, unsigned long long *hi_orig,
                                unsigned long long *keyA, uint32_t *valA, uint32_t *sh) {
  for (int i = threadIdx.x; i < kPasses * kRadix; i += blockDim.x) sh[i] = 0;
  __syncthreads();
  const int ub = bit_width(*reinterpret_cast<volatile uint32_t *>(&counts->max_bound));
  const bool unsorted = *reinterpret_cast<volatile uint32_t *>(&counts->unsorted) != 0;
  const bool wide = dbits + 1 + ub > 32;
  const int n_hi = (dbits + 1 + ub + 7) / 8;
  constexpr int kU = 4;  // entries per thread per round, loads issued together
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x * kU;
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x * kU; i0 < N; i0 += stride) {
    int32_t d[kU], u[kU], ar[kU], w[kU];
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + q * blockDim.x + threadIdx.x;
      const bool ok = i < N;
      d[q] = ok ? __ldg(dec + i) : 0;
      u[q] = ok ? __ldg(bound + i) : 0;
      ar[q] = ok ? __ldg(arrival + i) : 0;
      w[q] = ok ? __ldg(wait + i) : 0;
    }
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int64_t i = i0 + q * blockDim.x + threadIdx.x;
      const bool valid = i < N;
      unsigned long long key = 0;
      uint32_t a = 0;
      if (valid) {
        const int32_t dd = d[q] < 0 || d[q] >= D ? 0 : d[q];  // out-of-domain entries were flagged
        const int32_t uu = u[q] < 0 ? 0 : u[q];
        const int32_t aa = ar[q] < 0 ? 0 : ar[q];
        const bool promoted = w[q] > max_wait;
        const unsigned long long prim = promoted ? 0ull : static_cast<unsigned long long>(uu);
        key = (static_cast<unsigned long long>(dd) << (1 + ub)) |
              (static_cast<unsigned long long>(promoted ? 0u : 1u) << ub) | prim;
        a = static_cast<uint32_t>(aa);
        hi_orig[i] = key;
        if (unsorted) {
          keyA[i] = a;
          valA[i] = static_cast<uint32_t>(i);
        }
      }
      if (unsorted)
#pragma unroll
        for (int p = 0; p < kLoPasses; ++p) warp_count(sh + p * kRadix, (a >> (8 * p)) & 255u, valid);
      for (int p = 0; p < n_hi; ++p)
        warp_count(sh + (kLoPasses + p) * kRadix, static_cast<int>((key >> (8 * p)) & 255u), valid);
    }
  }
  (void)wide;
  __syncthreads();
  for (int i = threadIdx.x; i < kPasses * kRadix; i += blockDim.x) {
    const uint32_t c = sh[i];
    if (c) atomicAdd(&(&counts->h[0][0])[i], c);
  }
}

// Pass 2: keys in the compact layout and the histograms of every digit.
__global__ void __launch_bounds__(512)
order_keys_kernel(int64_t N, int D, int dbits, int64_t chunk, int Dp,
                  const int32_t *__restrict__ dec, const int32_t *__restrict__ bound,
                  const int32_t *__restrict__ wait, const int32_t *__restrict__ arrival,
                  int32_t max_wait, OrderCounts *counts, unsigned long long *hi_orig,
                  unsigned long long *keyA, uint32_t *valA, const int64_t *seg_off,
                  uint32_t *dec_cursor, const uint32_t *blk, const uint32_t *grp) {
  pdl_prologue();
  if (*reinterpret_cast<volatile uint32_t *>(&counts->segmented)) {
    // Each entry's segment key (not promoted, primary, index) goes to a slot
    // of its decoder's segment (hi_orig holds the segments).  A round of kU
    // entries per thread issues its loads and its slot claims together.
    constexpr int kU = kKeysU;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int ub = bit_width(*reinterpret_cast<volatile uint32_t *>(&counts->max_bound));
    const int ib = index_bits(N);
    auto seg_key = [&](int64_t i, int32_t u, int32_t w) {
      const unsigned long long np = w > max_wait ? 0ull : 1ull;
      const unsigned long long prim = np ? static_cast<unsigned long long>(u < 0 ? 0 : u) : 0ull;
      return (np << (ub + ib)) | (prim << ib) | static_cast<unsigned long long>(i);
    };
    if (*reinterpret_cast<volatile uint32_t *>(&counts->stable)) {
      // Stable: this block's range, round by round in index order.  An entry's
      // slot is its block's start in the segment, plus the entries of its
      // decoder in earlier rounds and earlier warps of this round, plus its
      // rank in its warp (item-major, then lane).
      extern __shared__ __align__(16) uint32_t ksm[];
      uint32_t *hw = ksm;                 // [warps][Dp] counts, then slot bases
      uint32_t *run = ksm + kPassWarps * Dp;  // [Dp] next slot of each decoder
      {
        // this block's first slot in every segment: seg_off[d] plus the
        // counts of the blocks before it, as the totals of the earlier groups
        // of kGroupBlocks blocks plus the rows of the earlier blocks of its
        // own group.  Thread (quad q of decoders, row group r) sums rows r,
        // r + rg, ... of that list; the row groups meet in hw.
        const int nq = Dp / 4;
        // rg row groups fit in hw: rg * Dp <= kPassWarps * Dp words
        const int rg = min(kPassWarps, max(1, static_cast<int>(blockDim.x) / nq));
        const int qd = threadIdx.x % nq, r = threadIdx.x / nq;
        const int g = static_cast<int>(blockIdx.x) / kGroupBlocks, b0 = g * kGroupBlocks;
        const int nrows = g + static_cast<int>(blockIdx.x) - b0;
        uint4 a0 = make_uint4(0, 0, 0, 0), a1 = a0;
        if (r < rg) {
          const uint4 *gcol = reinterpret_cast<const uint4 *>(grp) + qd;
          const uint4 *bcol = reinterpret_cast<const uint4 *>(blk) + static_cast<int64_t>(b0 - g) * nq + qd;
          auto row = [&](int i) { return i < g ? gcol[static_cast<int64_t>(i) * nq] : bcol[static_cast<int64_t>(i) * nq]; };
          int b2 = r;
          for (; b2 + rg < nrows; b2 += 2 * rg) {  // two loads in flight
            const uint4 v = row(b2), u = row(b2 + rg);
            a0.x += v.x, a0.y += v.y, a0.z += v.z, a0.w += v.w;
            a1.x += u.x, a1.y += u.y, a1.z += u.z, a1.w += u.w;
          }
          if (b2 < nrows) {
            const uint4 v = row(b2);
            a0.x += v.x, a0.y += v.y, a0.z += v.z, a0.w += v.w;
          }
          reinterpret_cast<uint4 *>(hw)[r * nq + qd] =
              make_uint4(a0.x + a1.x, a0.y + a1.y, a0.z + a1.z, a0.w + a1.w);
        }
        __syncthreads();
        for (int k = threadIdx.x; k < D; k += blockDim.x) {
          uint32_t v = static_cast<uint32_t>(seg_off[k]);
          for (int rr = 0; rr < rg; ++rr) v += hw[rr * Dp + k];
          run[k] = v;
        }
        __syncthreads();  // hw is zeroed next
      }
      const int64_t r_begin = static_cast<int64_t>(blockIdx.x) * chunk;
      const int64_t r_end = r_begin + chunk < N ? r_begin + chunk : N;
      for (int64_t i0 = r_begin; i0 < r_end; i0 += kKeysRound) {
        for (int k = threadIdx.x; k < kPassWarps * Dp; k += blockDim.x) hw[k] = 0;
        int d[kU];
        unsigned long long key[kU];
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const int64_t i = i0 + warp * (32 * kU) + q * 32 + lane;
          const bool ok = i < r_end;
          d[q] = ok ? __ldg(dec + i) : -1;
          if (ok && (d[q] < 0 || d[q] >= D)) d[q] = 0;  // out-of-domain entries were flagged
          key[q] = ok ? seg_key(i, __ldg(bound + i), __ldg(wait + i)) : 0ull;
        }
        __syncthreads();  // counts zeroed
        uint32_t rk[kU], base[kU];  // leader lane << 8 | rank in the group; group size, then base
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const unsigned pe = __match_any_sync(0xffffffffu, d[q]);
          const int leader = __ffs(pe) - 1;
          rk[q] = (static_cast<uint32_t>(leader) << 8) | static_cast<uint32_t>(__popc(pe & lanemask_lt()));
          base[q] = lane == leader ? static_cast<uint32_t>(__popc(pe)) : 0u;
        }
#pragma unroll
        for (int q = 0; q < kU; ++q)  // in item order, so ranks follow the index
          if (d[q] >= 0 && base[q] != 0) base[q] = atomicAdd(&hw[warp * Dp + d[q]], base[q]);
        __syncthreads();
        for (int k = threadIdx.x; k < D; k += blockDim.x) {  // exclusive over the warps
          uint32_t r = run[k];
          for (int w = 0; w < kPassWarps; ++w) {
            const uint32_t c = hw[w * Dp + k];
            hw[w * Dp + k] = r;
            r += c;
          }
          run[k] = r;
        }
        __syncthreads();
#pragma unroll
        for (int q = 0; q < kU; ++q) {
          const uint32_t b = __shfl_sync(0xffffffffu, base[q], static_cast<int>(rk[q] >> 8));
          if (d[q] >= 0) hi_orig[hw[warp * Dp + d[q]] + b + (rk[q] & 255u)] = key[q];
        }
        __syncthreads();  // the counts are zeroed again for the next round
      }
      return;
    }
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x * kU;
    for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x * kU; i0 < N; i0 += stride) {
      int d[kU];
      unsigned long long key[kU];
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const int64_t i = i0 + q * blockDim.x + threadIdx.x;
        d[q] = i < N ? __ldg(dec + i) : -1;
        if (i < N && (d[q] < 0 || d[q] >= D)) d[q] = 0;  // out-of-domain entries were flagged
        key[q] = i < N ? seg_key(i, __ldg(bound + i), __ldg(wait + i)) : 0ull;
      }
      uint32_t slot[kU];
      unsigned peers[kU];
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        peers[q] = __match_any_sync(0xffffffffu, d[q]);
        slot[q] = 0;
        if (d[q] >= 0 && lane == __ffs(peers[q]) - 1)
          slot[q] = atomicAdd(&dec_cursor[d[q]], static_cast<uint32_t>(__popc(peers[q])));
      }
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const uint32_t base = __shfl_sync(0xffffffffu, slot[q], __ffs(peers[q]) - 1);
        if (d[q] >= 0) hi_orig[seg_off[d[q]] + base + __popc(peers[q] & lanemask_lt())] = key[q];
      }
    }
    return;
  }
  __shared__ uint32_t sh[kPasses * kRadix];
  global_key_pass(N, D, dbits, dec, bound, wait, arrival, max_wait, counts, hi_orig, keyA, valA, sh);
}

// One block: digit offsets, active passes, buffer assignment, and the
// decoder segment offsets.
__device__ void plan_block(int64_t N, int D, int dbits, const OrderCounts *counts, OrderPlan *plan,
                           const uint32_t *dec_count, int64_t *seg_off) {
  __shared__ uint32_t s_warp[kRadix / 32];
  __shared__ long long s_w64[kRadix / 32];
  __shared__ int s_trivial[kPasses];
  __shared__ long long s_carry;
  const int b = threadIdx.x, lane = b & 31, warp = b >> 5;
  const bool act = b < kRadix;  // one thread per digit; the rest only meet the barriers
  uint32_t cnt[kPasses];  // all loads first
#pragma unroll
  for (int p = 0; p < kPasses; ++p) cnt[p] = act ? counts->h[p][b] : 0u;
#pragma unroll
  for (int p = 0; p < kPasses; ++p) {
    const uint32_t c = cnt[p];
    uint32_t incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (act && lane == 31) s_warp[warp] = incl;
    const int triv = __syncthreads_or(act && (static_cast<int64_t>(c) == N || N == 0));
    if (act) {
      uint32_t base = 0;
      for (int w = 0; w < warp; ++w) base += s_warp[w];
      plan->digit_off[p][b] = base + incl - c;
    }
    if (b == 0) s_trivial[p] = triv;
    __syncthreads();
  }
  if (b == 0) {
    const bool unsorted = counts->unsorted != 0;
    const int ub = counts->max_bound ? 32 - __clz(counts->max_bound) : 0;
    const int n_hi = min(kHiPasses, (dbits + 1 + ub + 7) / 8);
    plan->ubits = ub;
    plan->wide = dbits + 1 + ub > 32;
    int last = -1, n = 0, buf = kBufA;  // buffer holding the current keys
    for (int p = 0; p < kPasses; ++p) {
      plan->active[p] = 0;
      plan->shift[p] = p < kLoPasses ? 8 * p : 8 * (p - kLoPasses);
    }
    plan->gather_buf = -1;
    if (N > 0) {
      if (unsorted)
        for (int p = 0; p < kLoPasses; ++p) {
          if (s_trivial[p]) continue;
          plan->active[p] = 1;
          plan->src[p] = buf;
          plan->dst[p] = buf ^ 1;
          buf ^= 1;
          last = p;
          ++n;
        }
      const bool lo_ran = n > 0;
      if (lo_ran) plan->gather_buf = buf;
      bool first_hi = true;
      for (int p = kLoPasses; p < kLoPasses + n_hi; ++p) {
        if (s_trivial[p]) continue;
        plan->active[p] = 1;
        if (first_hi && !lo_ran) {
          plan->src[p] = kHiIdentity;
          plan->dst[p] = kBufA;
          buf = kBufA;
        } else {
          plan->src[p] = buf;
          plan->dst[p] = buf ^ 1;
          buf ^= 1;
        }
        first_hi = false;
        last = p;
        ++n;
      }
      if (last >= 0) plan->dst[last] = kPermOut;
    }
    plan->npasses = n;
    for (int p = 0, o = 0; p < kPasses; ++p) plan->ordinal[p] = plan->active[p] ? o++ : -1;
    s_carry = 0;
  }
  __syncthreads();
  // seg_off = exclusive scan of the per-decoder counts
  for (int base = 0; base <= D; base += kRadix) {
    const int k = base + b;
    const long long c = act && k < D ? dec_count[k] : 0;
    long long incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (act && lane == 31) s_w64[warp] = incl;
    __syncthreads();
    long long wb = 0;
    for (int w = 0; w < warp && act; ++w) wb += s_w64[w];
    const long long carry = s_carry;
    if (act && k <= D) seg_off[k] = carry + wb + incl - c;
    __syncthreads();
    if (b == kRadix - 1) s_carry = carry + wb + incl;
    __syncthreads();
  }
}

// The segment sort's digits are 9 bits wide.  Each per-warp counter word
// holds two 16-bit bins (2j low, 2j + 1 high): every count and position is at
// most kSegMax + a warp's items, so no half carries into the other.
constexpr int kSegBits = 9;
constexpr int kSegBins = 1 << kSegBits;
static_assert(2 * kSegMax + 32 * kSegIPT < 65536, "16-bit bins");
struct SegSmem {
  unsigned long long key[2][kSegMax];
  uint32_t hw[kSegWarps][kSegBins / 2];  // per-warp bin counts, then positions (packed pairs)
  uint32_t scan_w[kSegBins / 2 / 32];
  unsigned long long orv[kSegWarps], andv[kSegWarps];
};

// Stable LSD passes over the keys sm.key[cur][0, n) on the 9-bit digits of
// bits [lo_bit, nbits), skipping digits that are the same in every key (diff
// holds the bits that differ between the keys); returns the buffer holding
// the sorted keys.  All threads of the block take part.
__device__ int seg_lsd(SegSmem &sm, int n, unsigned long long diff, int lo_bit, int nbits, int cur) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int shift = lo_bit; shift < nbits; shift += kSegBits) {
    if (((diff >> shift) & (kSegBins - 1)) == 0) continue;  // same digit everywhere: order unchanged
    for (int i = tid; i < kSegWarps * kSegBins / 2; i += kSegThreads) (&sm.hw[0][0])[i] = 0;
    __syncthreads();
    // rank within the warp, stable in item order (warp-major, then item, then
    // lane): every match first, then one shared atomic per group leader,
    // issued in item order, whose old value gives the group's base
    uint32_t dr[kSegIPT];    // digit << 16 | leader lane << 8 | rank in the group
    uint32_t base[kSegIPT];  // the leader's group size, then the group's base
#pragma unroll
    for (int it = 0; it < kSegIPT; ++it) {
      const int x = warp * (32 * kSegIPT) + it * 32 + lane;
      const int d = x < n ? static_cast<int>((sm.key[cur][x] >> shift) & (kSegBins - 1)) : kSegBins;
      const unsigned pe = __match_any_sync(0xffffffffu, d);
      const int leader = __ffs(pe) - 1;
      dr[it] = (static_cast<uint32_t>(d) << 16) | (static_cast<uint32_t>(leader) << 8) |
               static_cast<uint32_t>(__popc(pe & lanemask_lt()));
      base[it] = lane == leader ? static_cast<uint32_t>(__popc(pe)) : 0u;
    }
#pragma unroll
    for (int it = 0; it < kSegIPT; ++it) {
      const int d = static_cast<int>(dr[it] >> 16);
      if (d < kSegBins && base[it] != 0) {
        const int h = (d & 1) * 16;
        base[it] = (atomicAdd(&sm.hw[warp][d >> 1], base[it] << h) >> h) & 0xffffu;
      }
    }
#pragma unroll
    for (int it = 0; it < kSegIPT; ++it)
      dr[it] = (dr[it] & 0xffff0000u) +
               __shfl_sync(0xffffffffu, base[it], static_cast<int>((dr[it] >> 8) & 31u)) +
               (dr[it] & 255u);
    __syncthreads();
    // per bin pair: exclusive scan over the warps (packed), then the bins'
    // starts from a block scan of the pair totals
    constexpr int kPairs = kSegBins / 2;
    uint32_t run = 0, tot = 0;
    if (tid < kPairs) {
      for (int w = 0; w < kSegWarps; ++w) {
        const uint32_t c = sm.hw[w][tid];
        sm.hw[w][tid] = run;
        run += c;
      }
      tot = (run & 0xffffu) + (run >> 16);
    }
    uint32_t incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (tid < kPairs && lane == 31) sm.scan_w[warp] = incl;
    __syncthreads();
    if (tid < kPairs) {
      uint32_t wb = 0;
      for (int w = 0; w < warp; ++w) wb += sm.scan_w[w];
      const uint32_t start0 = wb + incl - tot;           // bin 2j
      const uint32_t start1 = start0 + (run & 0xffffu);  // bin 2j + 1
      const uint32_t add = start0 | (start1 << 16);
      for (int w = 0; w < kSegWarps; ++w) sm.hw[w][tid] += add;
    }
    __syncthreads();
#pragma unroll
    for (int it = 0; it < kSegIPT; ++it) {
      const int x = warp * (32 * kSegIPT) + it * 32 + lane;
      if (x < n) {
        const int d = static_cast<int>(dr[it] >> 16);
        const uint32_t pos = (sm.hw[warp][d >> 1] >> ((d & 1) * 16)) & 0xffffu;
        sm.key[cur ^ 1][pos + (dr[it] & 0xffffu)] = sm.key[cur][x];
      }
    }
    __syncthreads();
    cur ^= 1;
  }
  return cur;
}

// The bits that differ between the keys sm.key[cur][0, n).
__device__ unsigned long long seg_diff(SegSmem &sm, int n, int cur) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  unsigned long long orv = 0, andv = ~0ull;
  for (int x = tid; x < n; x += kSegThreads) {
    orv |= sm.key[cur][x];
    andv &= sm.key[cur][x];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    orv |= __shfl_xor_sync(0xffffffffu, orv, o);
    andv &= __shfl_xor_sync(0xffffffffu, andv, o);
  }
  __syncthreads();  // orv / andv of an earlier call have been read
  if (lane == 0) {
    sm.orv[warp] = orv;
    sm.andv[warp] = andv;
  }
  __syncthreads();
  unsigned long long o = 0, a = ~0ull;
  for (int w = 0; w < kSegWarps; ++w) {
    o |= sm.orv[w];
    a &= sm.andv[w];
  }
  return o ^ a;
}

// Small calls (1 <= N <= kSegMax entries, D <= kSmallOrderD): the whole
// order in one block.  When arrival is non-decreasing along the index, one
// sort of (decoder, not promoted, promoted ? 0 : bound, index) gives the
// queue order.  Otherwise, when (decoder, not promoted, promoted ? 0 : bound,
// arrival, index) fits 64 bits (the bit widths taken from the largest
// arrival and the largest non-promoted bound), one sort on that key does;
// else the entries are put in arrival order first (a sort of (arrival,
// index)) and the first key's index is replaced by the arrival position.  Up
// to kBitonicN entries the sorts are bitonic networks over unique keys (a
// few dozen barrier-separated stages); larger calls take stable 9-bit LSD
// passes with the index in the keys' low bits.  The segment offsets come
// from binary searches over the sorted decoders.  One launch instead of a
// memset and four.
constexpr int kSmallOrderD = 4096;
constexpr int kBitonicN = 1024;

// Ascending bitonic sort of a[0, P) in shared memory, P a power of two (the
// block's threads take the compare-exchanges of each stage in turn).
template <typename T>
__device__ void block_bitonic(T *a, int P) {
  for (int k = 2; k <= P; k <<= 1)
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < P; i += blockDim.x) {
        const int l = i ^ j;
        if (l > i) {
          const T x = a[i], y = a[l];
          if ((x > y) == ((i & k) == 0)) {
            a[i] = y;
            a[l] = x;
          }
        }
      }
      __syncthreads();
    }
}

__global__ void __launch_bounds__(kSegThreads, 1)
order_small_kernel(int N, int D, int dbits, const int32_t *__restrict__ dec,
                   const int32_t *__restrict__ bound, const int32_t *__restrict__ wait,
                   const int32_t *__restrict__ arrival, int32_t max_wait, int32_t *perm,
                   int64_t *seg_off, int32_t *status) {
  pdl_prologue();
  extern __shared__ __align__(16) unsigned char small_raw[];
  SegSmem &sm = *reinterpret_cast<SegSmem *>(small_raw);
  __shared__ uint32_t s_amax, s_umax;
  const int tid = threadIdx.x;
  const int ib = index_bits(N);
  const unsigned long long imask = (1ull << ib) - 1;
  bool bad = false, unsorted = false;
  const bool bit = N <= kBitonicN;
  if (tid == 0) {
    s_amax = 0;
    s_umax = 0;
  }
  // the bitonic path's two key arrays sit back to back (the launch asks for
  // only 2 kBitonicN keys of shared memory then)
  unsigned long long *kb[2] = {reinterpret_cast<unsigned long long *>(small_raw),
                               reinterpret_cast<unsigned long long *>(small_raw) + kBitonicN};
  unsigned long long *k0 = bit ? kb[0] : sm.key[0];
  __syncthreads();
  uint32_t amax = 0;
  for (int x = tid; x < N; x += kSegThreads) {
    const int32_t a = __ldg(arrival + x);
    if (a < 0) bad = true;
    if (x + 1 < N && __ldg(arrival + x + 1) < a) unsorted = true;
    amax = max(amax, static_cast<uint32_t>(a < 0 ? 0 : a));
    k0[x] = (static_cast<unsigned long long>(a < 0 ? 0 : a) << ib) | static_cast<unsigned>(x);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) amax = max(amax, __shfl_xor_sync(0xffffffffu, amax, off));
  if ((tid & 31) == 0) atomicMax(&s_amax, amax);
  unsorted = __syncthreads_or(unsorted) != 0;
  // arrival out of index order: when (decoder, not promoted, primary,
  // arrival, index) fits 64 bits, one sort on that key gives the order;
  // otherwise the entries are put in arrival order first
  int ab = 0, ub = 0;
  bool one = false;
  if (unsorted) {
    uint32_t umax = 0;  // the largest bound of a non-promoted entry
    for (int x = tid; x < N; x += kSegThreads) {
      const int32_t u = __ldg(bound + x), w = __ldg(wait + x);
      if (w <= max_wait && u > 0) umax = max(umax, static_cast<uint32_t>(u));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) umax = max(umax, __shfl_xor_sync(0xffffffffu, umax, off));
    if ((tid & 31) == 0) atomicMax(&s_umax, umax);
    __syncthreads();
    ab = bit_width(s_amax);
    ub = bit_width(s_umax);
    one = dbits + 1 + ub + ab + ib <= 64;
  }
  int P = 1;
  while (P < N) P <<= 1;
  int cur = 0;
  const unsigned long long *ks;  // the sorted queue keys
  int dshift;                    // where their decoder field starts
  if (one) {
    for (int x = tid; x < N; x += kSegThreads) {  // each thread rewrites its own keys
      const int32_t a = __ldg(arrival + x), u = __ldg(bound + x), w = __ldg(wait + x);
      int32_t d = __ldg(dec + x);
      if (d < 0 || d >= D) {
        bad = true;
        d = 0;
      }
      if (u < 0) bad = true;
      const unsigned long long np = w > max_wait ? 0ull : 1ull;
      const unsigned long long prim = np ? static_cast<unsigned long long>(u < 0 ? 0 : u) : 0ull;
      unsigned long long key = (static_cast<unsigned long long>(d) << 1) | np;
      key = (key << ub) | prim;
      key = (key << ab) | static_cast<unsigned long long>(a < 0 ? 0 : a);
      k0[x] = (key << ib) | static_cast<unsigned>(x);
    }
    if (bit) {
      for (int x = N + tid; x < P; x += kSegThreads) k0[x] = ~0ull;
      __syncthreads();
      block_bitonic(k0, P);
      ks = k0;
    } else {
      __syncthreads();
      cur = seg_lsd(sm, N, seg_diff(sm, N, 0), ib, ib + ab + ub + 1 + dbits, 0);
      ks = sm.key[cur];
    }
    for (int t = tid; t < N; t += kSegThreads) perm[t] = static_cast<int32_t>(ks[t] & imask);
    dshift = ib + ab + ub + 1;
  } else {
    // k0 holds (arrival, index) keys, written before the barrier above
    if (unsorted) {
      if (bit) {
        for (int x = N + tid; x < P; x += kSegThreads) kb[0][x] = ~0ull;
        __syncthreads();
        block_bitonic(kb[0], P);
      } else {
        cur = seg_lsd(sm, N, seg_diff(sm, N, 0), ib, ib + 31, 0);
      }
    }
    unsigned long long *kin = bit ? kb[0] : sm.key[cur];
    unsigned long long *kout = bit ? kb[1] : sm.key[cur ^ 1];
    for (int t = tid; t < N; t += kSegThreads) {  // the queue keys, in arrival order
      const int x = static_cast<int>(kin[t] & imask);
      int32_t d = __ldg(dec + x);
      const int32_t u = __ldg(bound + x), w = __ldg(wait + x);
      if (d < 0 || d >= D) {
        bad = true;
        d = 0;
      }
      if (u < 0) bad = true;
      const unsigned long long np = w > max_wait ? 0ull : 1ull;
      const unsigned long long prim = np ? static_cast<unsigned long long>(u < 0 ? 0 : u) : 0ull;
      // low bits: the arrival position for the bitonic sort (unique keys), the
      // index for the stable passes
      kout[t] = (((static_cast<unsigned long long>(d) << 32) | (np << 31) | prim) << ib) |
                static_cast<unsigned>(bit ? t : x);
    }
    if (bit) {
      for (int t = N + tid; t < P; t += kSegThreads) kout[t] = ~0ull;
      __syncthreads();
      block_bitonic(kout, P);
      for (int t = tid; t < N; t += kSegThreads)  // arrival position -> index
        perm[t] = static_cast<int32_t>(kin[kout[t] & imask] & imask);
      ks = kout;
    } else {
      __syncthreads();
      cur ^= 1;
      cur = seg_lsd(sm, N, seg_diff(sm, N, cur), ib, ib + 32 + dbits, cur);
      for (int t = tid; t < N; t += kSegThreads) perm[t] = static_cast<int32_t>(sm.key[cur][t] & imask);
      ks = sm.key[cur];
    }
    dshift = ib + 32;
  }
  for (int d = tid; d <= D; d += kSegThreads) {  // entries of decoders below d
    int lo = 0, hi = N;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (static_cast<long long>(ks[mid] >> dshift) < d)
        lo = mid + 1;
      else
        hi = mid;
    }
    seg_off[d] = lo;
  }
  if (__syncthreads_or(bad) && tid == 0) flag_error(status, MAPS_E_RANGE);
}

// The bucketed form's inputs to the segment sort (on = 0: the entries are
// already in their segments).
struct BucketView {
  int on;
  const int32_t *item_dec;   // [item] decoder
  const int64_t *seg_off;    // [D + 1] segment offsets
  const uint32_t *blk, *bst; // [nblk][Dp] counts and bucket starts per bucketing block
  int64_t chunk;             // entries per bucketing block
  int Dp, nblk;
  // the global form's key pass, when arrival is out of index order
  int D, dbits;
  const int32_t *dec, *bound, *wait, *arrival;
  int32_t max_wait;
  unsigned long long *keyA;
  uint32_t *valA;
};

// Segmented form, step 2: each sort item (one decoder's queue, at most
// kSegMax entries) is sorted by one block on its keys (not promoted,
// promoted ? 0 : bound, index) with stable 9-bit LSD passes in shared
// memory, skipping digits that do not vary, and its indices are written.
// After a stable scatter the keys of a queue are already in index order and
// the index digits are skipped too.  In the bucketed form the item's entries
// are gathered from the bucketing blocks' buckets, in index order as well.
// Blocks take items in turn until none is left.
__global__ void __launch_bounds__(kSegThreads, 2)
order_segsort_kernel(int64_t N, OrderCounts *counts, const int64_t *item_off,
                     const int32_t *item_n, unsigned long long *seg_keys, int32_t *perm,
                     unsigned long long *run_keys, BucketView bv) {
  pdl_prologue();
  extern __shared__ __align__(16) unsigned char seg_raw[];
  if (bv.on && !counts->segmented) {
    // arrival is out of index order: the global form's key pass runs here
    global_key_pass(N, bv.D, bv.dbits, bv.dec, bv.bound, bv.wait, bv.arrival, bv.max_wait, counts,
                    seg_keys, bv.keyA, bv.valA, reinterpret_cast<uint32_t *>(seg_raw));
    return;
  }
  if (!counts->segmented) return;
  SegSmem &sm = *reinterpret_cast<SegSmem *>(seg_raw);
  // bucketed: the item's decoder's non-empty buckets, in block order: the
  // entries before each, and where it starts
  __shared__ uint32_t s_P[kPrepBlocks];
  __shared__ long long s_src[kPrepBlocks];
  __shared__ uint32_t s_pw[kSegWarps], s_nw[kSegWarps];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ub = counts->max_bound ? 32 - __clz(counts->max_bound) : 0;
  const int ib = index_bits(N);
  const int nbits = 1 + ub + ib;  // <= 1 + 31 + 31
  const int lo_bit = counts->stable ? ib : 0;  // first digit that needs sorting
  const int nitems = static_cast<int>(counts->nitems);
  for (int item = blockIdx.x; item < nitems; item += gridDim.x) {
    const int64_t off = item_off[item];
    const bool chunk = item_n[item] < 0;  // a chunk of a long queue: keys for the merges
    const int n = chunk ? -item_n[item] : item_n[item];
    unsigned long long orv = 0, andv = ~0ull;
    if (bv.on) {
      // Gather: the item is positions [o0, o0 + n) of its decoder's entries,
      // which the bucketing blocks hold in turn (block b: P[b] of them come
      // before it, in its bucket at bst[b][d]).
      const int d = bv.item_dec[item];
      const uint32_t o0 = static_cast<uint32_t>(off - bv.seg_off[d]);
      const bool blk_ok = tid < bv.nblk;
      const uint32_t c = blk_ok ? bv.blk[static_cast<int64_t>(tid) * bv.Dp + d] : 0u;
      const uint32_t st0 = blk_ok ? bv.bst[static_cast<int64_t>(tid) * bv.Dp + d] : 0u;
      // exclusive scans of the counts and of the non-empty flags over the blocks
      uint32_t incl = c;
      const unsigned ne = __ballot_sync(0xffffffffu, c > 0);
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (lane == 31) {
        s_pw[warp] = incl;
        s_nw[warp] = __popc(ne);
      }
      __syncthreads();
      uint32_t wb = 0, nb0 = 0, nruns = 0;
      for (int w = 0; w < kSegWarps; ++w) {
        wb += w < warp ? s_pw[w] : 0u;
        nb0 += w < warp ? s_nw[w] : 0u;
        nruns += s_nw[w];
      }
      if (c > 0) {
        const uint32_t r = nb0 + __popc(ne & lanemask_lt());
        s_P[r] = wb + incl - c;
        s_src[r] = static_cast<long long>(tid) * bv.chunk + st0;
      }
      __syncthreads();
#pragma unroll
      for (int it = 0; it < kSegIPT; ++it) {
        const int x = it * kSegThreads + tid;
        if (x < n) {
          const uint32_t pos = o0 + static_cast<uint32_t>(x);
          int lo = 0, hi = static_cast<int>(nruns) - 1;  // the last run with P <= pos
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_P[mid] <= pos)
              lo = mid;
            else
              hi = mid - 1;
          }
          const unsigned long long r = seg_keys[s_src[lo] + (pos - s_P[lo])];
          // r = not promoted << 63 | primary << 32 | index
          const unsigned long long key = ((r >> 63) << (ub + ib)) | (((r >> 32) & 0x7fffffffull) << ib) |
                                         (r & 0xffffffffull);
          sm.key[0][x] = key;
          orv |= key;
          andv &= key;
        }
      }
    } else {
#pragma unroll
      for (int it = 0; it < kSegIPT; ++it) {
        const int x = it * kSegThreads + tid;
        if (x < n) {
          const unsigned long long key = seg_keys[off + x];
          sm.key[0][x] = key;
          orv |= key;
          andv &= key;
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      orv |= __shfl_xor_sync(0xffffffffu, orv, o);
      andv &= __shfl_xor_sync(0xffffffffu, andv, o);
    }
    if (lane == 0) {
      sm.orv[warp] = orv;
      sm.andv[warp] = andv;
    }
    __syncthreads();
    unsigned long long diff = 0;
    {
      unsigned long long o = 0, a = ~0ull;
      for (int w = 0; w < kSegWarps; ++w) {
        o |= sm.orv[w];
        a &= sm.andv[w];
      }
      diff = o ^ a;  // bits that differ between keys of this segment
    }
    const int cur = seg_lsd(sm, n, diff, lo_bit, nbits, 0);
    const unsigned long long imask = (1ull << ib) - 1;
    if (chunk)
      for (int x = tid; x < n; x += kSegThreads) run_keys[off + x] = sm.key[cur][x];
    else
      for (int x = tid; x < n; x += kSegThreads) perm[off + x] = static_cast<int32_t>(sm.key[cur][x] & imask);
    __syncthreads();  // the next item reuses shared memory
  }
}

// Segmented form, step 3: merge level `level` of the long queues.  Runs of
// L = kSegMax << level sorted keys are merged pairwise from buf[level & 1]
// into buf[(level + 1) & 1], except at a queue's last level, which writes its
// indices to the order; a queue needing fewer levels is left alone.
// One block writes one tile of kMergeTile outputs: a merge-path search splits
// the two runs at the tile's ends, the tile's inputs are staged in shared
// memory, and each thread merges kMergeTile / kMergeThreads outputs after a
// second search.  Keys are unique, so there are no ties.
__device__ __forceinline__ int merge_path(const unsigned long long *A, int la,
                                          const unsigned long long *B, int lb, int d) {
  int lo = d > lb ? d - lb : 0, hi = d < la ? d : la;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (A[mid] < B[d - 1 - mid])
      lo = mid + 1;
    else
      hi = mid;
  }
  return lo;  // outputs before d taken from A
}

// All merge levels and the final order in one cooperative launch: the grid
// waits at a grid-wide barrier after each level.
// merge_path computed by one warp over global memory: each round probes 32
// diagonal positions at once and keeps the bracket between the last probe
// that takes from A and the first that does not, so a long run costs a few
// rounds of loads instead of one dependent load per halving.
__device__ __forceinline__ int merge_path_warp(const unsigned long long *A, int la,
                                               const unsigned long long *B, int lb, int d) {
  const int lane = threadIdx.x & 31;
  int lo = d > lb ? d - lb : 0, hi = d < la ? d : la;  // the answer lies in [lo, hi]
  while (hi - lo > 32) {
    const int span = hi - lo;
    const int pos = lo + static_cast<int>((static_cast<long long>(lane + 1) * span) / 33);
    const unsigned t = __ballot_sync(0xffffffffu, A[pos] < B[d - 1 - pos]);
    const int nt = __popc(t);  // probes before the answer
    const int plo = __shfl_sync(0xffffffffu, pos, nt > 0 ? nt - 1 : 0);
    const int phi = __shfl_sync(0xffffffffu, pos, nt < 32 ? nt : 31);
    lo = nt > 0 ? plo + 1 : lo;
    hi = nt < 32 ? phi : hi;
  }
  const int pos = lo + lane;
  const bool take_a = pos < hi && A[pos] < B[d - 1 - pos];
  return lo + __popc(__ballot_sync(0xffffffffu, take_a));
}

__device__ void merge_level(int level, int ntiles, const int64_t *mt_off, const int32_t *mt_n,
                            const int32_t *mt_t, unsigned long long *bufA,
                            unsigned long long *bufB, int32_t *perm, unsigned long long imask) {
  __shared__ unsigned long long s_a[kMergeTile], s_b[kMergeTile];
  __shared__ int s_split[2];
  const unsigned long long *src = (level & 1) ? bufB : bufA;
  unsigned long long *dst = (level & 1) ? bufA : bufB;
  const int64_t L = static_cast<int64_t>(kSegMax) << level;
  for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const int n = mt_n[tile];
    if (level >= merge_levels(n)) continue;  // this queue is complete (uniform per block)
    const int64_t off = mt_off[tile];
    const int w0 = mt_t[tile] * kMergeTile, w1 = min(w0 + kMergeTile, n);
    const int64_t pstart = (w0 / (2 * L)) * (2 * L);
    const int64_t rest = n - pstart;  // entries from this pair's start to the queue's end
    const int la = static_cast<int>(rest < L ? rest : L);
    const int lb = static_cast<int>(rest > L ? (rest < 2 * L ? rest : 2 * L) - L : 0);
    const unsigned long long *A = src + off + pstart, *B = A + la;
    const int d0 = static_cast<int>(w0 - pstart), d1 = static_cast<int>(w1 - pstart);
    if (threadIdx.x < 64) {  // warp 0 splits at d0, warp 1 at d1
      const int r = merge_path_warp(A, la, B, lb, threadIdx.x < 32 ? d0 : d1);
      if ((threadIdx.x & 31) == 0) s_split[threadIdx.x >> 5] = r;
    }
    __syncthreads();
    const int i0 = s_split[0], i1 = s_split[1];
    const int j0 = d0 - i0, j1 = d1 - i1;
    const int na = i1 - i0, nbb = j1 - j0;
    for (int x = threadIdx.x; x < na; x += kMergeThreads) s_a[x] = A[i0 + x];
    for (int x = threadIdx.x; x < nbb; x += kMergeThreads) s_b[x] = B[j0 + x];
    __syncthreads();
    constexpr int kPer = kMergeTile / kMergeThreads;
    const int dt = threadIdx.x * kPer;
    if (dt < na + nbb) {
      int ia = merge_path(s_a, na, s_b, nbb, dt), ib = dt - ia;
      // the queue's last level writes its order, the others the next runs
      const bool last = level == merge_levels(n) - 1;
      unsigned long long *out = dst + off + pstart + d0;
      int32_t *pout = perm + off + pstart + d0;
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        if (dt + q >= na + nbb) break;
        const bool takeA = ib >= nbb || (ia < na && s_a[ia] < s_b[ib]);
        const unsigned long long k = takeA ? s_a[ia++] : s_b[ib++];
        if (last)
          pout[dt + q] = static_cast<int32_t>(k & imask);
        else
          out[dt + q] = k;
      }
    }
    __syncthreads();  // the next tile reuses shared memory
  }
}

// The pairwise-ranked long queues: pair counts, a grid barrier, then every
// key to its place.  Runs are the segment sort's sorted chunks in keys.
__device__ void pair_rank_all(int64_t N, const OrderCounts *counts, const PairQueues &pq,
                              const unsigned long long *keys, int32_t *perm,
                              unsigned long long *sB, GridBar *bar, int32_t *status) {
  const int nq = static_cast<int>(counts->npairq);
  const int64_t npairs = min(static_cast<int64_t>(counts->npairs), pq.budget);
  // (1) pair p = (queue q, runs A != B): for each key of A, the keys of B below it
  for (int64_t p = blockIdx.x; p < npairs; p += gridDim.x) {
    int q = -1;
    for (int i = 0; i < nq; ++i) {  // the queue holding pair p (few queues)
      const int C = static_cast<int>((pq.n[i] + kSegMax - 1) / kSegMax);
      if (p >= pq.pair0[i] && p < pq.pair0[i] + static_cast<int64_t>(C) * (C - 1)) q = i;
    }
    if (q < 0) continue;  // a reservation no queue kept (uniform per block)
    const int64_t off = pq.off[q];
    const int n = pq.n[q], C = (n + kSegMax - 1) / kSegMax;
    const int l = static_cast<int>(p - pq.pair0[q]);
    const int A = l / (C - 1), b = l % (C - 1), B = b < A ? b : b + 1;
    const int nA = min(kSegMax, n - A * kSegMax), nB = min(kSegMax, n - B * kSegMax);
    const unsigned long long *rA = keys + off + static_cast<int64_t>(A) * kSegMax;
    const unsigned long long *rB = keys + off + static_cast<int64_t>(B) * kSegMax;
    for (int x = threadIdx.x; x < nB; x += blockDim.x) sB[x] = rB[x];
    __syncthreads();
    uint16_t *out = pq.cnt + p * kSegMax;
    for (int x = threadIdx.x; x < nA; x += blockDim.x) {
      const unsigned long long key = rA[x];
      int lo = 0, hi = nB;  // keys of B below key
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (sB[mid] < key)
          lo = mid + 1;
        else
          hi = mid;
      }
      out[x] = static_cast<uint16_t>(lo);
    }
    __syncthreads();  // sB serves the next pair
  }
  if (!grid_barrier(bar, status, g_lookback_spins)) return;
  // (2) each key's place: its place in its run plus its counts in the others
  const unsigned long long imask = (1ull << index_bits(N)) - 1;
  const int64_t gstride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int q = 0; q < nq; ++q) {
    const int64_t off = pq.off[q];
    const int n = pq.n[q], C = (n + kSegMax - 1) / kSegMax;
    const int64_t pair0 = pq.pair0[q];
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n; e += gstride) {
      const int A = static_cast<int>(e / kSegMax), x = static_cast<int>(e - static_cast<int64_t>(A) * kSegMax);
      int64_t pos = x;
      for (int B = 0; B < C; ++B) {
        if (B == A) continue;
        const int64_t pid = pair0 + static_cast<int64_t>(A) * (C - 1) + (B < A ? B : B - 1);
        pos += pq.cnt[pid * kSegMax + x];
      }
      perm[off + pos] = static_cast<int32_t>(keys[off + e] & imask);
    }
  }
}

__device__ void merge_all(int64_t N, const OrderCounts *counts, const int64_t *mt_off,
                          const int32_t *mt_n, const int32_t *mt_t, unsigned long long *bufA,
                          unsigned long long *bufB, int32_t *perm, GridBar *bar,
                          int32_t *status) {
  const int ntiles = static_cast<int>(counts->nmtiles);
  const int levels = static_cast<int>(counts->max_levels);
  const unsigned long long imask = (1ull << index_bits(N)) - 1;
  for (int level = 0; level < levels; ++level) {
    merge_level(level, ntiles, mt_off, mt_n, mt_t, bufA, bufB, perm, imask);
    if (level + 1 < levels && !grid_barrier(bar, status, g_lookback_spins)) return;
  }
}

struct PassSmem {
  unsigned long long keys[kTile];
  uint32_t vals[kTile];
  uint32_t hw[kPassWarps][kRadix];  // per-warp counts, then per-warp bin bases
  uint32_t tile_cnt[kRadix];
  uint32_t bin_start[kRadix];       // tile-local start of each bin
  uint32_t excl[kRadix];            // offset of this tile within each bin
  uint32_t scan_w[kRadix / 32];
  int tile;
};

// Key access for a pass: lo passes read arrival as 32 bits from a 64-bit
// slot array; narrow hi passes read 32-bit keys; wide ones 64-bit keys.
template <bool WIDE>
__device__ __forceinline__ unsigned long long load_key(const unsigned long long *k, int64_t i, bool lo) {
  if (lo) return k[i];
  if (WIDE) return k[i];
  return reinterpret_cast<const uint32_t *>(k)[i];
}
template <bool WIDE>
__device__ __forceinline__ void store_key(unsigned long long *k, int64_t i, unsigned long long v, bool lo) {
  if (lo || WIDE)
    k[i] = v;
  else
    reinterpret_cast<uint32_t *>(k)[i] = static_cast<uint32_t>(v);
}

// One tile of pass p: takes the next ticket; false when the pass has no tile
// left (the same answer in every thread).
template <bool WIDE>
__device__ bool order_pass_body(int p, int64_t N, const OrderPlan *plan, unsigned long long *keyA,
                                unsigned long long *keyB, uint32_t *valA, uint32_t *valB,
                                const unsigned long long *hi_orig, int32_t *perm,
                                unsigned long long *state, int64_t tiles, uint32_t *ticket,
                                int32_t *status, PassSmem &sm) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool lo = p < kLoPasses;
  const int src = plan->src[p], dst = plan->dst[p];
  const int shift = plan->shift[p];
  const bool identity = src == kHiIdentity;
  const unsigned long long *kin = src == kBufA ? keyA : (src == kBufB ? keyB : hi_orig);
  const uint32_t *vin = src == kBufA ? valA : valB;
  unsigned long long *kout = dst == kBufA ? keyA : keyB;
  uint32_t *vout = dst == kBufA ? valA : (dst == kBufB ? valB : reinterpret_cast<uint32_t *>(perm));
  const bool keys_out = dst != kPermOut;

  for (int i = tid; i < kPassWarps * kRadix; i += kPassThreads) (&sm.hw[0][0])[i] = 0;
  if (tid == 0) sm.tile = static_cast<int>(atomicAdd(ticket, 1u));
  __syncthreads();
  const int tile = sm.tile;
  if (tile >= tiles) return false;
  const int64_t base = static_cast<int64_t>(tile) * kTile;

  // load (all loads first), then rank within the warp (stable: warp-major,
  // then item, then lane)
  unsigned long long key[kIPT];
  uint32_t val[kIPT];
  int dig[kIPT];
  uint32_t rank[kIPT];
#pragma unroll
  for (int it = 0; it < kIPT; ++it) {
    const int64_t idx = base + warp * (32 * kIPT) + it * 32 + lane;
    const bool valid = idx < N;
    // the first hi pass reads the original keys in their own width
    key[it] = valid ? (identity ? (WIDE ? hi_orig[idx] : static_cast<uint32_t>(hi_orig[idx]))
                                : load_key<WIDE>(kin, idx, lo))
                    : 0ull;
    val[it] = valid ? (identity ? static_cast<uint32_t>(idx) : vin[idx]) : 0u;
    dig[it] = valid ? static_cast<int>((key[it] >> shift) & 255u) : kRadix;
  }
#pragma unroll
  for (int it = 0; it < kIPT; ++it) {
    const unsigned peers = __match_any_sync(0xffffffffu, dig[it]);
    const uint32_t before = __popc(peers & lanemask_lt());
    const bool valid = dig[it] < kRadix;
    uint32_t cur = 0;
    if (valid) cur = sm.hw[warp][dig[it]];
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) sm.hw[warp][dig[it]] = cur + __popc(peers);
    __syncwarp();
    rank[it] = cur + before;
  }
  __syncthreads();
  // Per bin: exclusive scan over warps and the tile total.  Then decoupled
  // look-back, one thread per bin: the tile publishes its aggregate, walks
  // back over its predecessors' (flag, count) words until it meets an
  // inclusive prefix, and publishes its own inclusive prefix.  Words carry the
  // flag in their top two bits.  Active pass number o uses state buffer o & 1
  // and clears this tile's row of the other buffer for active pass o + 1
  // (the buffer of the first active pass is cleared before the passes).
  const int ord = plan->ordinal[p];
  unsigned long long *st_cur = state + static_cast<size_t>(ord & 1) * tiles * kRadix;
  unsigned long long *st_nxt = state + static_cast<size_t>((ord + 1) & 1) * tiles * kRadix;
  if (tid < kRadix) {
    uint32_t run = 0;
    for (int w = 0; w < kPassWarps; ++w) {
      const uint32_t c = sm.hw[w][tid];
      sm.hw[w][tid] = run;
      run += c;
    }
    sm.tile_cnt[tid] = run;
    const size_t me = static_cast<size_t>(tile) * kRadix + tid;
    const bool publish = tile != g_withheld_tile;  // always, outside the test aid
    const uint32_t spin_limit = g_lookback_spins;
    st_nxt[me] = 0ull;
    if (publish)
      st_release_u64(&st_cur[me], static_cast<unsigned long long>(run) |
                                      (static_cast<unsigned long long>(tile == 0 ? kFlagInc : kFlagAgg) << 62));
    unsigned long long excl = 0;
    if (tile > 0) {
      for (int q = tile - 1;; --q) {
        unsigned long long v;
        uint32_t spins = 0;
        while (((v = ld_acquire_u64(&st_cur[static_cast<size_t>(q) * kRadix + tid])) >> 62) == 0) {
          if (++spins > spin_limit) {
            // give up: count the rest as empty.  The offsets then only come
            // out smaller than the true ones, so every write of the pass
            // stays inside [0, N); the order is wrong and the call reports it.
            flag_error(status, MAPS_E_TIMEOUT);
            v = static_cast<unsigned long long>(kFlagInc) << 62;
            break;
          }
          __nanosleep(32);
        }
        excl += v & ((1ull << 62) - 1);
        if ((v >> 62) == kFlagInc || q == 0) break;
      }
      if (publish)
        st_release_u64(&st_cur[me], (excl + run) | (static_cast<unsigned long long>(kFlagInc) << 62));
    }
    sm.excl[tid] = static_cast<uint32_t>(excl);
  }
  __syncthreads();
  // tile-local bin starts (the first 8 warps hold the 256 bins)
  uint32_t bc = 0, bincl = 0;
  if (tid < kRadix) {
    bc = sm.tile_cnt[tid];
    bincl = bc;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, bincl, off);
      if (lane >= off) bincl += y;
    }
    if (lane == 31) sm.scan_w[warp] = bincl;
  }
  __syncthreads();
  if (tid < kRadix) {
    uint32_t wb = 0;
    for (int w = 0; w < warp; ++w) wb += sm.scan_w[w];
    sm.bin_start[tid] = wb + bincl - bc;
  }
  __syncthreads();
  // stage the tile in shared memory sorted by digit
#pragma unroll
  for (int it = 0; it < kIPT; ++it) {
    if (dig[it] < kRadix) {
      const uint32_t s = sm.bin_start[dig[it]] + sm.hw[warp][dig[it]] + rank[it];
      sm.keys[s] = key[it];
      sm.vals[s] = val[it];
    }
  }
  __syncthreads();
  const int64_t rem = N - base;
  const int n_tile = static_cast<int>(rem < kTile ? rem : kTile);
  for (int s = tid; s < n_tile; s += kPassThreads) {
    const unsigned long long k = sm.keys[s];
    const int d = static_cast<int>((k >> shift) & 255u);
    const uint32_t pos = plan->digit_off[p][d] + sm.excl[d] + (s - sm.bin_start[d]);
    if (keys_out) store_key<WIDE>(kout, pos, k, lo);
    vout[pos] = sm.vals[s];
  }
  __syncthreads();  // the next tile reuses shared memory
  return true;
}

// The last launch of every call, cooperative, so that its phases meet at grid
// barriers:
//   * segmented form: the merge levels of the long queues, if there are any;
//   * otherwise block 0 plans the global passes (digit offsets, active passes,
//     buffers, decoder segment offsets), then the passes run, one grid-wide
//     sweep each: a block takes tiles by ticket until none is left, so a
//     tile's look-back only waits on tiles already taken by running blocks.
//     With no active pass the identity is the order.
__global__ void __launch_bounds__(kPassThreads, 2)
order_finish_kernel(int n_hi, int64_t N, int D, int dbits, const OrderCounts *counts,
                    OrderPlan *plan, const uint32_t *dec_count, int64_t *seg_off,
                    const int64_t *mt_off, const int32_t *mt_n, const int32_t *mt_t,
                    PairQueues pq, unsigned long long *keyA, unsigned long long *keyB, uint32_t *valA,
                    uint32_t *valB, const unsigned long long *hi_orig, int32_t *perm,
                    unsigned long long *state, int64_t tiles, uint32_t *tickets, GridBar *bar,
                    int32_t *status) {
  pdl_prologue();
  if (static_cast<int>(blockIdx.x) == g_absent_block) return;  // test aid, normally -1
  // every block takes the same branches, so no block waits at a barrier alone;
  // a barrier that ran out (MAPS_E_TIMEOUT) ends the block at once
  if (*reinterpret_cast<const volatile uint32_t *>(&counts->segmented)) {
    if (counts->npairq > 0) {
      extern __shared__ __align__(16) unsigned char pair_raw[];
      pair_rank_all(N, counts, pq, keyA, perm, reinterpret_cast<unsigned long long *>(pair_raw), bar, status);
    }
    if (counts->nmtiles > 0) merge_all(N, counts, mt_off, mt_n, mt_t, keyA, keyB, perm, bar, status);
    return;
  }
  if (blockIdx.x == 0) plan_block(N, D, dbits, counts, plan, dec_count, seg_off);
  // the look-back words of the first active pass start at zero (the passes
  // clear the other buffer as they go)
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < tiles * kRadix;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    state[i] = 0ull;
  if (!grid_barrier(bar, status, g_lookback_spins)) return;
  const int npasses = plan->npasses;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  PassSmem &sm = *reinterpret_cast<PassSmem *>(smem_raw);
  const bool wide = plan->wide != 0;
  auto run_pass = [&](int p) {
    if (wide)
      while (order_pass_body<true>(p, N, plan, keyA, keyB, valA, valB, hi_orig, perm, state,
                                   tiles, tickets + p, status, sm)) {
      }
    else
      while (order_pass_body<false>(p, N, plan, keyA, keyB, valA, valB, hi_orig, perm, state,
                                    tiles, tickets + p, status, sm)) {
      }
    return grid_barrier(bar, status, g_lookback_spins);
  };
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t first = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (int p = 0; p < kLoPasses; ++p)
    if (plan->active[p] && !run_pass(p)) return;
  const int gb = plan->gather_buf;
  if (gb >= 0) {  // after arrival passes the keys follow the arrival order
    unsigned long long *k = gb == kBufA ? keyA : keyB;
    const uint32_t *v = gb == kBufA ? valA : valB;
    for (int64_t i = first; i < N; i += stride) {
      const unsigned long long x = hi_orig[v[i]];
      if (wide)
        k[i] = x;
      else
        reinterpret_cast<uint32_t *>(k)[i] = static_cast<uint32_t>(x);
    }
    if (!grid_barrier(bar, status, g_lookback_spins)) return;
  }
  for (int p = kLoPasses; p < kLoPasses + n_hi; ++p)
    if (plan->active[p] && !run_pass(p)) return;
  if (npasses == 0)
    for (int64_t i = first; i < N; i += stride) perm[i] = static_cast<int32_t>(i);
}

static_assert(sizeof(PassSmem) >= kSegMax * sizeof(unsigned long long),
              "one sorted run fits the finishing kernel's shared memory");

// Blocks of the finishing kernel that can be resident at once (its grid limit
// as a cooperative launch).
int64_t finish_grid(size_t smem) {
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, order_finish_kernel, kPassThreads,
                                                    smem) != cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  return static_cast<int64_t>(per_sm) * sm_count();
}

struct OrderWs {
  OrderCounts *counts;
  uint32_t *dec_count;
  uint32_t *dec_cursor;  // segmented form: slots taken per decoder
  uint32_t *tickets;
  GridBar *bar;  // the finishing kernel's grid barrier
  unsigned long long *state;  // [2][tiles][256] look-back words (buffer 0 zeroed by the finishing kernel)
  size_t zero_bytes;  // counts .. tickets are contiguous and zeroed per call
  OrderPlan *plan;
  int64_t *item_off;  // sort items: queues and chunks of long queues
  int32_t *item_n;
  int32_t *item_dec;
  int64_t *mt_off;    // merge tiles of the long queues
  int32_t *mt_n, *mt_t;
  int64_t nitems_max, ntiles_max;
  PairQueues pq;      // pairwise-ranked long queues
  unsigned long long *hi_orig, *keyA, *keyB;
  uint32_t *valA, *valB;
  uint32_t *blk;      // stable scatter: [blocks][Dp] counts per prep block
  uint32_t *bst;      // bucketed form: [blocks][Dp] each block's bucket starts
  uint32_t *grp;      // stable scatter: [groups][Dp] counts per kGroupBlocks prep blocks (zeroed)
  int64_t chunk;      // entries per prep / key block
  int blocks, Dp;
};

OrderWs carve_order(Carve &c, int64_t N, int D) {
  OrderWs w;
  const int64_t tiles = std::max<int64_t>(1, (N + kTile - 1) / kTile);
  const size_t zero_begin = (c.off + kAlign - 1) / kAlign * kAlign;
  w.counts = c.take<OrderCounts>(1);
  w.dec_count = c.take<uint32_t>(static_cast<size_t>(D));
  w.dec_cursor = c.take<uint32_t>(static_cast<size_t>(D));
  w.chunk = D <= kStableD ? bucket_chunk(N) : prep_chunk(N);  // bucketed form: whole rounds
  w.blocks = static_cast<int>(std::max<int64_t>(1, (N + w.chunk - 1) / w.chunk));
  w.Dp = (D + 3) / 4 * 4;
  w.grp = c.take<uint32_t>(D <= kStableD ? static_cast<size_t>((w.blocks + kGroupBlocks - 1) / kGroupBlocks) * w.Dp
                                         : 1);
  w.tickets = c.take<uint32_t>(kPasses);
  w.bar = c.take<GridBar>(1);
  w.zero_bytes = c.off - zero_begin;
  w.state = c.take<unsigned long long>(static_cast<size_t>(2) * tiles * kRadix);
  w.plan = c.take<OrderPlan>(1);
  w.nitems_max = D + N / kSegMax + 1;
  w.ntiles_max = N / kMergeTile + D + 1;
  w.item_off = c.take<int64_t>(static_cast<size_t>(w.nitems_max));
  w.item_n = c.take<int32_t>(static_cast<size_t>(w.nitems_max));
  w.item_dec = c.take<int32_t>(static_cast<size_t>(w.nitems_max));
  w.mt_off = c.take<int64_t>(static_cast<size_t>(w.ntiles_max));
  w.mt_n = c.take<int32_t>(static_cast<size_t>(w.ntiles_max));
  w.mt_t = c.take<int32_t>(static_cast<size_t>(w.ntiles_max));
  w.pq.budget = pair_budget(N);
  const size_t nq_max = static_cast<size_t>(w.pq.budget / 2 + 1);  // a queue has >= 2 pairs
  w.pq.off = c.take<int64_t>(nq_max);
  w.pq.n = c.take<int32_t>(nq_max);
  w.pq.pair0 = c.take<int32_t>(nq_max);
  w.pq.cnt = c.take<uint16_t>(static_cast<size_t>(w.pq.budget) * kSegMax + 1);
  const size_t n = static_cast<size_t>(N > 0 ? N : 1);
  w.hi_orig = c.take<unsigned long long>(n);
  w.keyA = c.take<unsigned long long>(n);
  w.keyB = c.take<unsigned long long>(n);
  w.valA = c.take<uint32_t>(n);
  w.valB = c.take<uint32_t>(n);
  w.blk = c.take<uint32_t>(D <= kStableD ? static_cast<size_t>(w.blocks) * w.Dp : 1);
  w.bst = c.take<uint32_t>(D <= kStableD ? static_cast<size_t>(w.blocks) * w.Dp : 1);
  return w;
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_order_local_workspace_size(int64_t N, int32_t D) {
  maps::Carve c(nullptr);
  maps::carve_order(c, N < 0 ? 0 : N, D < 1 ? 1 : D);
  return c.bytes();
}

int maps_order_local(int64_t N, int32_t D, const int32_t *dec, const int32_t *bound,
                     const int32_t *wait, const int32_t *arrival, int32_t max_wait,
                     int32_t *perm_out, int64_t *seg_off_out, void *ws, size_t ws_bytes,
                     void *stream) {
  using namespace maps;
  if (N < 0 || N > 0x7fffffffLL || D < 1 || seg_off_out == nullptr) return MAPS_E_INVALID;
  if (N > 0 && (dec == nullptr || bound == nullptr || wait == nullptr || arrival == nullptr ||
                perm_out == nullptr))
    return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_order_local_workspace_size(N, D)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  Carve cv(ws);
  const OrderWs w = carve_order(cv, N, D);
  int dbits = 0;  // bits of the largest decoder index
  while ((1ll << dbits) < D) ++dbits;
  if (N >= 1 && N <= kSegMax && D <= kSmallOrderD) {
    const size_t small_smem =
        N <= kBitonicN ? 2 * kBitonicN * sizeof(unsigned long long) : sizeof(SegSmem);
    MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_small_kernel,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          static_cast<int>(sizeof(SegSmem)))));
    launch_pdl(order_small_kernel, 1, kSegThreads, small_smem, s, static_cast<int>(N), D, dbits, dec,
               bound, wait, arrival, max_wait, perm_out, seg_off_out, status);
    return launch_ok();
  }
  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.counts, 0, w.zero_bytes, s)));
  // hi passes that can be active: the key has at most dbits + 1 + 31 bits
  const int n_hi = std::min(kHiPasses, (dbits + 1 + 31 + 7) / 8);
  const int sms = sm_count();
  const int64_t tiles = std::max<int64_t>(1, (N + kTile - 1) / kTile);
  // D <= kStableD: one bucketing pass replaces the prep and key passes
  const bool bucketed = N > 0 && D <= kStableD;
  BucketView bv = {};
  if (bucketed) {
    const size_t bsmem = sizeof(uint32_t) * static_cast<size_t>(kPassWarps + 1) * w.Dp;
    MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_bucket_kernel,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          static_cast<int>(bsmem))));
    launch_pdl(order_bucket_kernel, w.blocks, 512, bsmem, s, N, D, w.chunk, w.Dp, dec, bound, wait,
               arrival, max_wait, w.counts, w.dec_count, status, seg_off_out, w.item_off, w.item_n,
               w.item_dec, w.mt_off, w.mt_n, w.mt_t, w.pq, w.blk, w.bst, w.hi_orig);
    bv.on = 1;
    bv.item_dec = w.item_dec;
    bv.seg_off = seg_off_out;
    bv.blk = w.blk;
    bv.bst = w.bst;
    bv.chunk = w.chunk;
    bv.Dp = w.Dp;
    bv.nblk = w.blocks;
    bv.D = D;
    bv.dbits = dbits;
    bv.dec = dec;
    bv.bound = bound;
    bv.wait = wait;
    bv.arrival = arrival;
    bv.max_wait = max_wait;
    bv.keyA = w.keyA;
    bv.valA = w.valA;
  } else if (N > 0) {
    launch_pdl(order_prep_kernel, w.blocks, 512, 0, s, N, D, w.chunk, dec, bound, wait, arrival,
               max_wait, w.counts, w.dec_count, status, seg_off_out, w.item_off, w.item_n,
               w.item_dec, w.mt_off, w.mt_n, w.mt_t, w.pq, w.blk, w.grp, w.Dp);
    // the stable scatter's per-warp counts and running slots
    const size_t keys_smem =
        D <= kStableD ? sizeof(uint32_t) * static_cast<size_t>(kPassWarps + 1) * w.Dp : 0;
    if (keys_smem > 0)
      MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_keys_kernel,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            static_cast<int>(keys_smem))));
    launch_pdl(order_keys_kernel, w.blocks, 512, keys_smem, s, N, D, dbits, w.chunk, w.Dp, dec,
               bound, wait, arrival, max_wait, w.counts, w.hi_orig, w.keyA, w.valA, seg_off_out,
               w.dec_cursor, w.blk, w.grp);
  }
  MAPS_TRY(launch_ok());
  if (N == 0) {  // no entries: the segment offsets are all zero
    MAPS_TRY(cuda_ok(cudaMemsetAsync(seg_off_out, 0, sizeof(int64_t) * (static_cast<size_t>(D) + 1), s)));
    return MAPS_OK;
  }
  const size_t seg_smem = sizeof(SegSmem);
  MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_segsort_kernel,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(seg_smem))));
  // (the bucketed form's segment sort may run the global key pass: at least
  // as many blocks as the bucketing pass)
  const int64_t seg_grid = std::min<int64_t>(bucketed ? std::max<int64_t>(w.nitems_max, w.blocks)
                                                      : w.nitems_max,
                                             2LL * sms);
  launch_pdl(order_segsort_kernel, static_cast<unsigned>(seg_grid), kSegThreads, seg_smem, s, N,
             w.counts, w.item_off, w.item_n, w.hi_orig, perm_out, w.keyA, bv);
  const size_t smem = sizeof(PassSmem);
  MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_finish_kernel,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(smem))));
  // the global passes take tiles by ticket, so any resident grid completes
  // them; the pairwise ranks take one block per pair
  MAPS_TRY(launch_coop(order_finish_kernel,
                       std::min<int64_t>(std::max<int64_t>(tiles, w.pq.budget), finish_grid(smem)),
                       kPassThreads, smem, s, n_hi, N, D, dbits, w.counts, w.plan, w.dec_count,
                       seg_off_out, w.mt_off, w.mt_n, w.mt_t, w.pq, w.keyA, w.keyB, w.valA, w.valB,
                       w.hi_orig, perm_out, w.state, tiles, w.tickets, w.bar, status));
  return launch_ok();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of maps_order_local.
//
// For callers that cannot allocate device memory at all -- code running
// where cudaMalloc is unavailable or forbidden, such as a scheduler embedded
// in a host process whose allocator is owned by someone else, or one that
// must never allocate after start-up -- the scratch lives in this file-scope
// device array instead of a caller workspace.  Every GPU that loads the
// library holds it until the process exits.
// ---------------------------------------------------------------------------
namespace maps {
namespace {

constexpr int64_t kStaticMaxN = 65536;  // entries
constexpr int32_t kStaticMaxD = 4096;   // decoders
constexpr size_t kStaticBytes = size_t(5) << 20;
static __device__ __align__(256) unsigned char g_order_scratch[kStaticBytes];

// Device address of the static scratch on the current device.  The host-side
// symbol is not a device address; the lookup is a cheap host call, made on
// every call so that a reset device or a new context is never handed an old
// address.  The first call on a device also loads the library's device code
// there if that has not happened yet.
int static_scratch(void **out) {
  void *p = nullptr;
  MAPS_TRY(cuda_ok(cudaGetSymbolAddress(&p, g_order_scratch)));
  if (p == nullptr || !aligned(p, kAlign)) return MAPS_E_CUDA;
  *out = p;
  return MAPS_OK;
}

}  // namespace
}  // namespace maps

extern "C" int maps_order_local_static(int64_t N, int32_t D, const int32_t *dec,
                                       const int32_t *bound, const int32_t *wait,
                                       const int32_t *arrival, int32_t max_wait,
                                       int32_t *perm_out, int64_t *seg_off_out,
                                       int32_t *status_host, void *stream) {
  using namespace maps;
  if (N < 0 || D < 1) return MAPS_E_INVALID;
  if (N > kStaticMaxN || D > kStaticMaxD) return MAPS_E_WORKSPACE;
  const size_t need = maps_order_local_workspace_size(N, D);
  if (need > kStaticBytes) return MAPS_E_WORKSPACE;
  void *ws = nullptr;
  MAPS_TRY(static_scratch(&ws));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents: start this call's status
  // at zero (the order itself zeroes every counter it needs)
  MAPS_TRY(cuda_ok(cudaMemsetAsync(ws, 0, kCtrlBytes, s)));
  MAPS_TRY(maps_order_local(N, D, dec, bound, wait, arrival, max_wait, perm_out, seg_off_out, ws,
                            kStaticBytes, stream));
  if (status_host != nullptr) {
    *status_host = maps_check(ws, stream);
    return *status_host;
  }
  return MAPS_OK;
}

extern "C" int maps_test_absent_block(int32_t block) {
  using namespace maps;
  MAPS_TRY(cuda_ok(cudaMemcpyToSymbol(g_absent_block, &block, sizeof(block))));
  return MAPS_OK;
}

extern "C" int maps_test_withhold_lookback(int32_t tile, uint32_t spin_limit) {
  using namespace maps;
  const uint32_t spins = spin_limit == 0 ? kSpinLimit : spin_limit;
  MAPS_TRY(cuda_ok(cudaMemcpyToSymbol(g_withheld_tile, &tile, sizeof(tile))));
  MAPS_TRY(cuda_ok(cudaMemcpyToSymbol(g_lookback_spins, &spins, sizeof(spins))));
  return MAPS_OK;
}
