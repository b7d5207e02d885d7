// occupancy.cu -- projected KV-token occupancy over the step horizon.
//
// K[k][t] = sum over residents r of decoder k with t < e_r of (b_r + t),
// b_r = p_r + g_r + 1, e_r = min(max(U_r - g_r, 1), H), which is
//   K[k][t] = SumB_k(t) + t * Cnt_k(t)
// with Cnt / SumB the count and b-sum of residents still live at t.
//
// Layout of the work.  A decoder's horizon is cut into tiles of W steps.
//   1. bucket kernel, one CTA per decoder: reads the decoder's residents
//      once, forms (b, e) and counting-sorts the pairs by the tile that holds
//      their last live step, into the workspace, with per-tile offsets and
//      per-tile carries (count and b-sum of the residents live past the
//      tile).  It also checks the inputs and that K[k][0] = sum of b fits
//      int32.
//   2. tile kernel, one CTA per (decoder, tile), launched tile-major: reads
//      its carry and the pairs of its own tile.  A tile with few pairs sums
//      them directly; a denser one bins them into a shared-memory end-step
//      histogram whose reverse scan, plus the carry, gives every cell's live
//      count and b-sum.  Cells are written through shared staging rows as
//      whole 128-byte lines.
// For horizons of more than kMaxTiles tiles a single-kernel form is used
// instead, in which every tile CTA streams all of its decoder's residents.
// Optionally every group of 16 steps also yields kmax[k][t/16] =
// max (K[k][t] + t), a summary the dispatch uses for the prefix maxima of
// earlier horizon tiles.
//
// Integer range: every resident is live at t = 0, so K[k][0] = sum of b_r
// and every partial sum is at most K[k][0]; if that total exceeds INT32_MAX
// the call reports MAPS_E_RANGE, otherwise the 32-bit shared-memory sums
// cannot wrap.  A thread forms its cells in 32 bits when a bound over its
// cells shows that none exceeds INT32_MAX, and exactly in 64 bits otherwise.
#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kOccThreads = 256;  // tile CTAs: 256 threads x CPT cells
constexpr int kWarps = kOccThreads / 32;
constexpr int kBucketThreads = 512;
constexpr int kBlock = 16;     // steps per kmax summary entry
constexpr int kPerThread = 4;  // entries a thread loads per round
constexpr int kRound = kPerThread * kOccThreads;
constexpr int kBucketRound = kPerThread * kBucketThreads;
constexpr int kMaxTiles = 128;  // tiles per decoder of the bucketed form
constexpr int kBHold = 8;       // residents a bucket thread keeps in registers
// A tile holding at most this many end steps skips the histogram: its pairs
// are kept as a list that every thread scans for its own cells.
constexpr int kSparse = 32;

// Per-warp carry partials and the block scan's scratch.
struct TileScan {
  uint32_t part[2][kWarps];  // per-warp carry partials (count, b-sum)
  uint32_t wsum[2][kWarps];
  uint32_t carry[2];
};

// Shared-memory end-step histogram of one tile (the long-horizon form).  Bins
// are padded by 4 words after every CPT bins so that the threads' 16-byte
// reads of their own CPT bins fall on distinct banks.
template <int CPT>
struct TileSmem {
  static constexpr int W = kOccThreads * CPT;
  static constexpr int kPad = CPT == 4 ? 0 : 4;
  static constexpr int WP = W + (W / CPT) * kPad;
  int32_t cnt[WP];  // bin j: residents whose last live step is t0 + j
  int32_t sb[WP];   // ... and the sum of their b
  TileScan scan;
};

// This warp's staging rows for the stores (32 lanes x (CPT + 4) words), over
// the count bins, which hold exactly the block's rows when CPT >= 8.
template <int CPT>
__device__ __forceinline__ uint32_t *stage_rows(TileSmem<CPT> &sm) {
  static_assert(CPT < 8 || TileSmem<CPT>::WP >= kOccThreads * (CPT + 4), "staging fits the bins");
  return reinterpret_cast<uint32_t *>(sm.cnt) + (threadIdx.x >> 5) * 32 * (CPT + 4);
}

template <int CPT>
__device__ __forceinline__ void zero_bins(TileSmem<CPT> &sm) {
  for (int i = threadIdx.x * 4; i < TileSmem<CPT>::WP; i += kOccThreads * 4) {
    *reinterpret_cast<int4 *>(&sm.cnt[i]) = make_int4(0, 0, 0, 0);
    *reinterpret_cast<int4 *>(&sm.sb[i]) = make_int4(0, 0, 0, 0);
  }
}

template <int CPT>
__device__ __forceinline__ void add_to_bin(TileSmem<CPT> &sm, int jj, int32_t b) {
  const int jp = jj + (jj / CPT) * TileSmem<CPT>::kPad;
  atomicAdd(&sm.cnt[jp], 1);
  atomicAdd(&sm.sb[jp], b);  // exact while sum b fits int32
}

// Writes the cells tid*CPT + c, c < CPT, of tile [t0, t0 + W) of row k.
// bc[c] / bs[c] are the count and b-sum of the residents whose last live step
// is that cell, tot_c / tot_s their sums over the thread's cells, and
// c_hi / s_hi the count and b-sum of the residents live past the thread's
// last cell.  The 32-bit sums only wrap when sum b exceeds INT32_MAX, which
// is reported as MAPS_E_RANGE.  Every thread of the block calls it.
template <int CPT, bool VEC>
__device__ __forceinline__ void write_cells(const uint32_t (&bc)[CPT], const uint32_t (&bs)[CPT],
                                            uint32_t tot_c, uint32_t tot_s, uint32_t c_hi,
                                            uint32_t s_hi, int H, int k, int t0, int32_t *K,
                                            uint32_t *kmax, int32_t *status, uint32_t *stage) {
  const int tid = threadIdx.x, lane = tid & 31;
  const int cell0 = t0 + tid * CPT;
  const uint32_t tc0 = static_cast<uint32_t>(cell0);
  int32_t *row = K + static_cast<int64_t>(k) * H;
  uint32_t bmax = 0;  // max of K + t over this thread's valid cells
  // Both running sums only grow towards the thread's first cell, so their
  // totals and the last cell's step bound every cell of the thread.
  const unsigned long long bound64 =
      static_cast<unsigned long long>(tc0 + CPT - 1) * (c_hi + tot_c) + (s_hi + tot_s);
  // every cell valid and exact in 32 bits
  const bool fast = VEC && cell0 + CPT <= H && bound64 <= 0x7fffffffull;
  uint32_t o[CPT];
  if (fast) {
    uint32_t run_c = c_hi, run_s = s_hi;
    if (tot_c == 0) {
      // no resident ends in these cells: K is affine in t over them, and
      // K + t grows with t, so the last cell holds the maximum
#pragma unroll
      for (int c = 0; c < CPT; ++c) o[c] = (tc0 + c) * run_c + run_s;
      bmax = o[CPT - 1] + tc0 + CPT - 1;
    } else {
#pragma unroll
      for (int c = CPT - 1; c >= 0; --c) {
        run_c += bc[c];
        run_s += bs[c];
        o[c] = (tc0 + c) * run_c + run_s;
        bmax = max(bmax, o[c] + tc0 + c);
      }
    }
  }
  if (CPT >= 8 && __all_sync(0xffffffffu, fast)) {
    // The warp's 32 * CPT cells are contiguous: pass them through this warp's
    // shared staging rows (CPT + 4 words a lane, so both the row writes and
    // the chunk reads spread over the banks) and store 512 contiguous bytes
    // per instruction, whole sectors instead of half sectors.
    constexpr int kLS = CPT + 4;
    constexpr int kChunks = CPT / 4;  // 16-byte chunks per lane
#pragma unroll
    for (int c = 0; c < kChunks; ++c)
      *reinterpret_cast<uint4 *>(stage + lane * kLS + 4 * c) =
          make_uint4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
    __syncwarp();
    int32_t *wrow = row + (cell0 - lane * CPT);  // the warp's first cell
#pragma unroll
    for (int s2 = 0; s2 < kChunks; ++s2) {
      const int q = s2 * 32 + lane;  // chunk of the warp's range
      const uint4 v = *reinterpret_cast<const uint4 *>(stage + (q / kChunks) * kLS + (q % kChunks) * 4);
      *reinterpret_cast<uint4 *>(wrow + 4 * q) = v;
    }
    __syncwarp();  // the staging rows are reused
  } else if (fast) {
#pragma unroll
    for (int c = 0; c < CPT; c += 4)
      *reinterpret_cast<int4 *>(row + cell0 + c) = make_int4(o[c], o[c + 1], o[c + 2], o[c + 3]);
  } else if (cell0 < H) {
    uint32_t run_c = c_hi, run_s = s_hi;
    bool over = false;
#pragma unroll
    for (int c = CPT - 1; c >= 0; --c) {
      run_c += bc[c];
      run_s += bs[c];
      if (cell0 + c < H) {
        const uint32_t t = tc0 + c;
        const unsigned long long v = static_cast<unsigned long long>(t) * run_c + run_s;
        over |= (v >> 31) != 0;
        const uint32_t ov = static_cast<uint32_t>(v);
        bmax = max(bmax, ov + t);
        row[cell0 + c] = static_cast<int32_t>(ov);
      }
    }
    if (over) flag_error(status, MAPS_E_RANGE);
  }
  if (kmax != nullptr) {
    constexpr int L = kBlock / CPT > 0 ? kBlock / CPT : 1;  // lanes per 16-step block
#pragma unroll
    for (int off = L / 2; off > 0; off >>= 1) bmax = max(bmax, __shfl_xor_sync(0xffffffffu, bmax, off));
    if ((lane % L) == 0 && cell0 < H) {
      const int64_t nb = (static_cast<int64_t>(H) + kBlock - 1) / kBlock;
      kmax[static_cast<int64_t>(k) * nb + cell0 / kBlock] = bmax;
    }
  }
}

// Writes tile [t0, t0 + W) of row k from every thread's own bins.  Entry:
// sc.part[][warp] written by every warp and a block barrier since.  Cell l
// needs every bin at or after l: the thread's own bins from l up, all bins of
// the threads above it (a block suffix scan), and the carry.
template <int CPT, bool VEC>
__device__ __forceinline__ void emit_cells(const uint32_t (&bc)[CPT], const uint32_t (&bs)[CPT],
                                           TileScan &sc, int H, int k, int t0, int32_t *K,
                                           uint32_t *kmax, int32_t *status, uint32_t *stage) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t tot_c = 0, tot_s = 0;
#pragma unroll
  for (int c = 0; c < CPT; ++c) {
    tot_c += bc[c];
    tot_s += bs[c];
  }
  uint32_t suf_c = tot_c, suf_s = tot_s;  // inclusive suffix within the warp
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t yc = __shfl_down_sync(0xffffffffu, suf_c, off);
    const uint32_t ys = __shfl_down_sync(0xffffffffu, suf_s, off);
    if (lane + off < 32) {
      suf_c += yc;
      suf_s += ys;
    }
  }
  if (lane == 0) {
    sc.wsum[0][warp] = suf_c;
    sc.wsum[1][warp] = suf_s;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive suffix over the warps' totals; the carry
    uint32_t wc = lane < kWarps ? sc.wsum[0][lane] : 0u;
    uint32_t ws = lane < kWarps ? sc.wsum[1][lane] : 0u;
    const uint32_t oc = wc, os = ws;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t yc = __shfl_down_sync(0xffffffffu, wc, off);
      const uint32_t ys = __shfl_down_sync(0xffffffffu, ws, off);
      if (lane + off < 32) {
        wc += yc;
        ws += ys;
      }
    }
    uint32_t cc = lane < kWarps ? sc.part[0][lane] : 0u;
    uint32_t cs = lane < kWarps ? sc.part[1][lane] : 0u;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      cc += __shfl_xor_sync(0xffffffffu, cc, off);
      cs += __shfl_xor_sync(0xffffffffu, cs, off);
    }
    __syncwarp();
    if (lane < kWarps) {
      sc.wsum[0][lane] = wc - oc;
      sc.wsum[1][lane] = ws - os;
    }
    if (lane == 0) {
      sc.carry[0] = cc;
      sc.carry[1] = cs;
    }
  }
  __syncthreads();

  const uint32_t c_hi = sc.carry[0] + sc.wsum[0][warp] + (suf_c - tot_c);
  const uint32_t s_hi = sc.carry[1] + sc.wsum[1][warp] + (suf_s - tot_s);
  write_cells<CPT, VEC>(bc, bs, tot_c, tot_s, c_hi, s_hi, H, k, t0, K, kmax, status, stage);
}

// The histogram form: each thread takes its own CPT bins into registers.
template <int CPT, bool VEC>
__device__ __forceinline__ void emit_tile(TileSmem<CPT> &sm, int H, int k, int t0, int32_t *K,
                                          uint32_t *kmax, int32_t *status) {
  constexpr int kPad = TileSmem<CPT>::kPad;
  const int32_t *cb = &sm.cnt[threadIdx.x * (CPT + kPad)], *sb = &sm.sb[threadIdx.x * (CPT + kPad)];
  uint32_t bc[CPT], bs[CPT];
#pragma unroll
  for (int c = 0; c < CPT; c += 4) {
    const int4 x = *reinterpret_cast<const int4 *>(cb + c);
    const int4 y = *reinterpret_cast<const int4 *>(sb + c);
    bc[c] = x.x, bc[c + 1] = x.y, bc[c + 2] = x.z, bc[c + 3] = x.w;
    bs[c] = y.x, bs[c + 1] = y.y, bs[c + 2] = y.z, bs[c + 3] = y.w;
  }
  // the staging rows reuse the count bins: every thread has read its own bins
  // before the scan's first barrier
  emit_cells<CPT, VEC>(bc, bs, sm.scan, H, k, t0, K, kmax, status, stage_rows(sm));
}

// Resident terms: false for a negative length (a range error).
__device__ __forceinline__ bool resident_terms(int32_t p, int32_t g, int32_t U, int H,
                                               int32_t &b32, int32_t &e, bool &big) {
  if ((p | g | U) < 0) return false;
  const long long b = static_cast<long long>(p) + g + 1;
  big = b > 0x7fffffffLL;  // alone already above the K[k][0] limit
  b32 = static_cast<int32_t>(big ? 0x7fffffffLL : b);
  e = U - g;  // both non-negative: no wrap
  e = e < 1 ? 1 : (e > H ? H : e);
  return true;
}

template <int NW>
__device__ __forceinline__ long long block_sum_ll(long long v, long long *s_red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  if (lane == 0) s_red[warp] = v;
  __syncthreads();
  long long t = 0;
  for (int w = 0; w < NW; ++w) t += s_red[w];
  return t;
}

// ---------------------------------------------------------------------------
// 1. Bucket kernel: one CTA per decoder.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kBucketThreads)
occ_bucket_kernel(int H, int T, int log2W, const int64_t *__restrict__ res_off, int64_t R,
                  const int32_t *__restrict__ prompt, const int32_t *__restrict__ gen,
                  const int32_t *__restrict__ bound, int2 *__restrict__ bucket,
                  int32_t *__restrict__ tile_off, uint2 *__restrict__ tile_carry,
                  int32_t *status) {
  pdl_prologue();
  __shared__ int s_cnt[kMaxTiles];
  __shared__ uint32_t s_sb[kMaxTiles];
  __shared__ int s_cur[kMaxTiles];
  __shared__ unsigned long long s_total;  // sum of b over the decoder's residents
  const int k = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
  int64_t lo = res_off[k], hi = res_off[k + 1];
  if (lo < 0 || hi < lo || hi > R || hi - lo > 0x7fffffffLL) {
    if (tid == 0) flag_error(status, MAPS_E_RANGE);
    lo = hi = 0;
  }
  const int n = static_cast<int>(hi - lo);
  const int32_t *pp = prompt + lo, *pg = gen + lo, *pu = bound + lo;
  if (tid < kMaxTiles) s_cnt[tid] = 0, s_sb[tid] = 0;
  if (tid == 0) s_total = 0;
  __syncthreads();

  // tile starts and carries (the residents live past each tile); T <= kMaxTiles
  auto publish = [&]() {
    if (tid == 0) {
      int run = 0;
      int32_t *to = tile_off + static_cast<int64_t>(k) * (T + 1);
      for (int y = 0; y < T; ++y) {
        to[y] = run;
        s_cur[y] = run;
        run += s_cnt[y];
      }
      to[T] = run;
    } else if (tid == 32) {
      uint32_t cc = 0, cs = 0;
      uint2 *tc = tile_carry + static_cast<int64_t>(k) * T;
      for (int y = T - 1; y >= 0; --y) {
        tc[y] = make_uint2(cc, cs);
        cc += static_cast<uint32_t>(s_cnt[y]);
        cs += s_sb[y];
      }
    } else if (tid == 64 && s_total > 0x7fffffffull) {
      flag_error(status, MAPS_E_RANGE);
    }
  };
  // a group of lanes with the same tile: count and b-sum to the tile's bins
  // (every lane of a group reduces over that group only; the b-sum wraps
  // only past INT32_MAX, which is reported)
  auto count = [&](int tile, int32_t b32, unsigned peers) {
    const uint32_t bsum = __reduce_add_sync(peers, tile >= 0 ? static_cast<uint32_t>(b32) : 0u);
    if (tile >= 0 && lane == __ffs(peers) - 1) {
      atomicAdd(&s_cnt[tile], __popc(peers));
      atomicAdd(&s_sb[tile], bsum);
    }
  };
  // ... and its slots in the tile's range of the bucket array
  auto scatter = [&](int tile, int32_t b32, int32_t e, unsigned peers) {
    const int leader = __ffs(peers) - 1;
    int base = 0;
    if (tile >= 0 && lane == leader) base = atomicAdd(&s_cur[tile], __popc(peers));
    base = __shfl_sync(0xffffffffu, base, leader);
    if (tile >= 0) bucket[lo + base + __popc(peers & ((1u << lane) - 1u))] = make_int2(b32, e);
  };
  auto add_total = [&](unsigned long long total) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) total += __shfl_xor_sync(0xffffffffu, total, off);
    if (lane == 0) atomicAdd(&s_total, total);
  };

  if (n <= kBHold * kBucketThreads) {
    // Held form: one read of the residents, kept in registers with their
    // peer masks through both passes.
    int32_t hb[kBHold], he[kBHold], tl[kBHold];
    unsigned pr[kBHold];
    bool bad = false;
    unsigned long long total = 0;
    {
      int32_t p[kBHold], g[kBHold], U[kBHold];
#pragma unroll
      for (int j = 0; j < kBHold; ++j) {
        const int i = j * kBucketThreads + tid;
        const bool ok = i < n;
        p[j] = ok ? __ldg(pp + i) : -1;
        g[j] = ok ? __ldg(pg + i) : 0;
        U[j] = ok ? __ldg(pu + i) : 0;
      }
#pragma unroll
      for (int j = 0; j < kBHold; ++j) {
        bool big = false;
        hb[j] = he[j] = 0;
        tl[j] = -1;
        if (resident_terms(p[j], g[j], U[j], H, hb[j], he[j], big)) {
          tl[j] = (he[j] - 1) >> log2W;
          total += static_cast<unsigned long long>(hb[j]);
          bad |= big;
        } else if (j * kBucketThreads + tid < n) {
          bad = true;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kBHold; ++j) {
      pr[j] = __match_any_sync(0xffffffffu, tl[j]);
      count(tl[j], hb[j], pr[j]);
    }
    add_total(total);
    if (bad) flag_error(status, MAPS_E_RANGE);
    __syncthreads();
    publish();
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kBHold; ++j) scatter(tl[j], hb[j], he[j], pr[j]);
    return;
  }

  // Streamed form (more residents than the registers hold): pass 1 counts,
  // pass 2 reads the residents again (from L2) and scatters.
  for (int r0 = 0; r0 < n; r0 += kBucketRound) {
    int32_t p[kPerThread], g[kPerThread], U[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const int i = r0 + j * kBucketThreads + tid;
      const bool ok = i < n;
      p[j] = ok ? __ldg(pp + i) : -1;
      g[j] = ok ? __ldg(pg + i) : 0;
      U[j] = ok ? __ldg(pu + i) : 0;
    }
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      int32_t b32, e;
      bool big;
      const int tile = resident_terms(p[j], g[j], U[j], H, b32, e, big) ? (e - 1) >> log2W : -1;
      count(tile, b32, __match_any_sync(0xffffffffu, tile));
    }
  }
  bool bad = false;
  unsigned long long total = 0;
  __syncthreads();
  for (int r0 = 0; r0 < n; r0 += kBucketRound) {  // totals and checks ride on pass 2
    int32_t p[kPerThread], g[kPerThread], U[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const int i = r0 + j * kBucketThreads + tid;
      const bool ok = i < n;
      p[j] = ok ? __ldg(pp + i) : -1;
      g[j] = ok ? __ldg(pg + i) : 0;
      U[j] = ok ? __ldg(pu + i) : 0;
    }
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      int32_t b32, e;
      bool big = false;
      if (resident_terms(p[j], g[j], U[j], H, b32, e, big)) {
        total += static_cast<unsigned long long>(b32);
        bad |= big;
      } else if (r0 + j * kBucketThreads + tid < n) {
        bad = true;
      }
    }
  }
  add_total(total);
  if (bad) flag_error(status, MAPS_E_RANGE);
  __syncthreads();
  publish();
  __syncthreads();
  for (int r0 = 0; r0 < n; r0 += kBucketRound) {
    int32_t p[kPerThread], g[kPerThread], U[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const int i = r0 + j * kBucketThreads + tid;
      const bool ok = i < n;
      p[j] = ok ? __ldg(pp + i) : -1;
      g[j] = ok ? __ldg(pg + i) : 0;
      U[j] = ok ? __ldg(pu + i) : 0;
    }
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      int32_t b32 = 0, e = 0;
      bool big;
      const int tile = resident_terms(p[j], g[j], U[j], H, b32, e, big) ? (e - 1) >> log2W : -1;
      scatter(tile, b32, e, __match_any_sync(0xffffffffu, tile));
    }
  }
}

// ---------------------------------------------------------------------------
// 2. Tile kernel: one CTA per (decoder, tile), reading the sorted pairs of its
// own tile and the tile's carry (count and b-sum of the residents live past
// it) from the bucket kernel.
// ---------------------------------------------------------------------------
template <int CPT, bool VEC>
__global__ void __launch_bounds__(kOccThreads, 4)
occ_tile_kernel(int H, int D, int T, const int64_t *__restrict__ res_off, int64_t R,
                const int2 *__restrict__ bucket, const int32_t *__restrict__ tile_off,
                const uint2 *__restrict__ tile_carry, int32_t *__restrict__ K,
                uint32_t *__restrict__ kmax, int32_t *status) {
  pdl_prologue();
  __shared__ __align__(16) TileSmem<CPT> sm;
  // tile-major order: the early tiles, where most residents end, start first
  const int ti = blockIdx.x / D, k = blockIdx.x - (blockIdx.x / D) * D;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t0 = ti * TileSmem<CPT>::W;
  int64_t lo = res_off[k];
  const int32_t *to = tile_off + static_cast<int64_t>(k) * (T + 1);
  const int a = to[ti], m = to[ti + 1];
  const uint2 car = tile_carry[static_cast<int64_t>(k) * T + ti];
  if (lo < 0 || lo > R) lo = 0;  // reported by the bucket kernel; the range is then empty
  const int2 *bk = bucket + lo;

  if (m - a <= kSparse) {  // the same for the whole block
    // Sparse tile: every thread reads the tile's few pairs (one address
    // across the warp).  A pair past the thread's last cell adds to every one
    // of its cells, one inside from its own cell down; no block scan needed.
    uint32_t c_hi = car.x, s_hi = car.y;
    uint32_t bc[CPT], bs[CPT];
#pragma unroll
    for (int c = 0; c < CPT; ++c) bc[c] = bs[c] = 0;
    uint32_t tot_c = 0, tot_s = 0;
    const int c0 = tid * CPT;
    for (int j = a; j < m; ++j) {
      const int2 v = __ldg(bk + j);
      const int q = v.y - 1 - t0 - c0;  // the pair's last live step, from the thread's first cell
      if (q >= CPT) {
        c_hi += 1;
        s_hi += static_cast<uint32_t>(v.x);
      } else if (q >= 0) {
        tot_c += 1;
        tot_s += static_cast<uint32_t>(v.x);
#pragma unroll
        for (int c = 0; c < CPT; ++c)
          if (q == c) {
            bc[c] += 1;
            bs[c] += static_cast<uint32_t>(v.x);
          }
      }
    }
    write_cells<CPT, VEC>(bc, bs, tot_c, tot_s, c_hi, s_hi, H, k, t0, K, kmax, status,
                          stage_rows(sm));
    return;
  }

  zero_bins(sm);
  __syncthreads();
  for (int r0 = a; r0 < m; r0 += kRound) {
    int2 v[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const int i = r0 + j * kOccThreads + tid;
      v[j] = i < m ? __ldg(bk + i) : make_int2(0, 0);
    }
#pragma unroll
    for (int j = 0; j < kPerThread; ++j)
      if (r0 + j * kOccThreads + tid < m) add_to_bin(sm, v[j].y - 1 - t0, v[j].x);
  }
  if (lane == 0) {  // the carry enters the scan as warp 0's partial
    sm.scan.part[0][warp] = warp == 0 ? car.x : 0u;
    sm.scan.part[1][warp] = warp == 0 ? car.y : 0u;
  }
  __syncthreads();
  emit_tile<CPT, VEC>(sm, H, k, t0, K, kmax, status);
}

// ---------------------------------------------------------------------------
// Long horizons: every tile CTA streams all of its decoder's residents.
// ---------------------------------------------------------------------------
template <int CPT, bool VEC>
__global__ void __launch_bounds__(kOccThreads, 4)
occ_direct_kernel(int H, int T, const int64_t *__restrict__ res_off, int64_t R,
                  const int32_t *__restrict__ prompt, const int32_t *__restrict__ gen,
                  const int32_t *__restrict__ bound, int32_t *__restrict__ K,
                  uint32_t *__restrict__ kmax, int32_t *status) {
  pdl_prologue();
  __shared__ __align__(16) TileSmem<CPT> sm;
  __shared__ long long s_red[kWarps];
  constexpr int W = TileSmem<CPT>::W;
  const int k = blockIdx.x / T, ti = blockIdx.x - (blockIdx.x / T) * T;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t0 = ti * W;
  int64_t lo = res_off[k], hi = res_off[k + 1];
  if (lo < 0 || hi < lo || hi > R) {
    if (tid == 0) flag_error(status, MAPS_E_RANGE);
    lo = hi = 0;
  }
  const int64_t n = hi - lo;
  const int32_t *pp = prompt + lo, *pg = gen + lo, *pu = bound + lo;
  zero_bins(sm);
  __syncthreads();

  bool bad = false;
  long long total = 0;
  uint32_t car_c = 0, car_s = 0;
  for (int64_t r0 = 0; r0 < n; r0 += kRound) {
    int32_t p[kPerThread], g[kPerThread], U[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const int64_t i = r0 + j * kOccThreads + tid;
      const bool ok = i < n;
      p[j] = ok ? __ldg(pp + i) : -1;
      g[j] = ok ? __ldg(pg + i) : 0;
      U[j] = ok ? __ldg(pu + i) : 0;
    }
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      int32_t b32, e;
      bool big;
      if (resident_terms(p[j], g[j], U[j], H, b32, e, big)) {
        total += b32;
        bad |= big;
        const int jj = e - 1 - t0;  // last live step, relative to the tile
        if (jj >= W) {
          car_c += 1;
          car_s += static_cast<uint32_t>(b32);
        } else if (jj >= 0) {
          add_to_bin(sm, jj, b32);
        }
      } else if (r0 + j * kOccThreads + tid < n) {
        bad = true;
      }
    }
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
  const long long sum_b = block_sum_ll<kWarps>(total, s_red);
  if (ti == 0 && tid == 0 && sum_b > 0x7fffffffLL) flag_error(status, MAPS_E_RANGE);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    car_c += __shfl_xor_sync(0xffffffffu, car_c, off);
    car_s += __shfl_xor_sync(0xffffffffu, car_s, off);
  }
  if (lane == 0) {
    sm.scan.part[0][warp] = car_c;
    sm.scan.part[1][warp] = car_s;
  }
  __syncthreads();
  emit_tile<CPT, VEC>(sm, H, k, t0, K, kmax, status);
}

struct OccPlan {
  int cpt, T, log2W;
  bool bucketed;
};

OccPlan plan_occ(int32_t H, int64_t R) {
  OccPlan p;
  p.cpt = H <= 1024 ? 4 : (H <= 2048 ? 8 : 16);
  p.log2W = 8 + (p.cpt == 4 ? 2 : (p.cpt == 8 ? 3 : 4));  // W = 256 threads x CPT
  p.T = static_cast<int>((static_cast<int64_t>(H) + (1 << p.log2W) - 1) >> p.log2W);
  p.bucketed = p.T <= kMaxTiles && R <= 0x7fffffffLL;
  return p;
}

size_t carve_occ(Carve &c, int32_t D, int64_t R, const OccPlan &p, int2 **bucket,
                 int32_t **tile_off, uint2 **tile_carry) {
  if (p.bucketed) {
    *bucket = c.take<int2>(static_cast<size_t>(R));
    *tile_off = c.take<int32_t>(static_cast<size_t>(D) * (p.T + 1));
    *tile_carry = c.take<uint2>(static_cast<size_t>(D) * p.T);
  }
  return c.bytes();
}

template <int CPT, bool VEC>
void launch_tiles(const OccPlan &p, int64_t blocks, cudaStream_t s, int H, const int64_t *res_off,
                  int64_t R, const int32_t *prompt, const int32_t *gen, const int32_t *bound,
                  const int2 *bucket, const int32_t *tile_off, const uint2 *tile_carry,
                  int32_t *K, uint32_t *kmax, int32_t *status) {
  const dim3 grid(static_cast<unsigned>(blocks));
  if (p.bucketed)
    launch_pdl(occ_tile_kernel<CPT, VEC>, grid, kOccThreads, 0, s, H, static_cast<int>(blocks / p.T), p.T, res_off, R, bucket,
               tile_off, tile_carry, K, kmax, status);
  else
    launch_pdl(occ_direct_kernel<CPT, VEC>, grid, kOccThreads, 0, s, H, p.T, res_off, R, prompt, gen,
                                                            bound, K, kmax, status);
}

template <int CPT>
void launch_cpt(bool vec, const OccPlan &p, int64_t blocks, cudaStream_t s, int H,
                const int64_t *res_off, int64_t R, const int32_t *prompt, const int32_t *gen,
                const int32_t *bound, const int2 *bucket, const int32_t *tile_off,
                const uint2 *tile_carry, int32_t *K, uint32_t *kmax, int32_t *status) {
  if (vec)
    launch_tiles<CPT, true>(p, blocks, s, H, res_off, R, prompt, gen, bound, bucket, tile_off,
                            tile_carry, K, kmax, status);
  else
    launch_tiles<CPT, false>(p, blocks, s, H, res_off, R, prompt, gen, bound, bucket, tile_off,
                             tile_carry, K, kmax, status);
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_project_occupancy_workspace_size(int32_t D, int32_t H, int64_t R) {
  using namespace maps;
  if (D < 1 || H < 1 || R < 0) return kCtrlBytes;
  Carve c(nullptr);
  int2 *bucket = nullptr;
  int32_t *tile_off = nullptr;
  uint2 *tile_carry = nullptr;
  return carve_occ(c, D, R, plan_occ(H, R), &bucket, &tile_off, &tile_carry);
}

int maps_project_occupancy(int32_t D, int32_t H, const int64_t *res_off, int64_t R,
                           const int32_t *prompt, const int32_t *gen, const int32_t *bound,
                           int32_t *K_out, uint32_t *kmax_out, void *ws, size_t ws_bytes,
                           void *stream) {
  using namespace maps;
  if (D < 1 || H < 1 || H > (1 << 28) || R < 0 || res_off == nullptr || K_out == nullptr)
    return MAPS_E_INVALID;
  if (R > 0 && (prompt == nullptr || gen == nullptr || bound == nullptr)) return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_project_occupancy_workspace_size(D, H, R)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  const OccPlan p = plan_occ(H, R);
  const int64_t blocks = static_cast<int64_t>(D) * p.T;
  if (blocks > 0x7fffffffLL) return MAPS_E_INVALID;
  Carve c(ws);
  int2 *bucket = nullptr;
  int32_t *tile_off = nullptr;
  uint2 *tile_carry = nullptr;
  carve_occ(c, D, R, p, &bucket, &tile_off, &tile_carry);
  if (p.bucketed) {
    launch_pdl(occ_bucket_kernel, D, kBucketThreads, 0, s, H, p.T, p.log2W, res_off, R, prompt,
               gen, bound, bucket, tile_off, tile_carry, status);
    MAPS_TRY(launch_ok());
  }
  const bool vec = (H % 4 == 0) && aligned(K_out, 16);
  if (p.cpt == 16)
    launch_cpt<16>(vec, p, blocks, s, H, res_off, R, prompt, gen, bound, bucket, tile_off, tile_carry, K_out,
                   kmax_out, status);
  else if (p.cpt == 8)
    launch_cpt<8>(vec, p, blocks, s, H, res_off, R, prompt, gen, bound, bucket, tile_off, tile_carry, K_out,
                  kmax_out, status);
  else
    launch_cpt<4>(vec, p, blocks, s, H, res_off, R, prompt, gen, bound, bucket, tile_off, tile_carry, K_out,
                  kmax_out, status);
  return launch_ok();
}

}  // extern "C"
