// order.cu -- local SJF reordering with max-wait promotion (Sec. 3.3).
//
// The queue order is the lexicographic order of
//     (decoder, not promoted, promoted ? arrival : bound, arrival, index)
// computed as a stable least-significant-digit radix sort of 8-bit digits:
//   * one upfront pass builds the 64-bit key (decoder << 32 | not-promoted
//     << 31 | primary), counts every digit of it and of the arrival, counts
//     entries per decoder, and checks whether arrival is already
//     non-decreasing in index;
//   * a one-block plan kernel turns the counts into digit offsets, marks a
//     digit pass inactive when every key has the same digit, and skips the
//     arrival passes when arrival is already in index order (stability then
//     gives the arrival tie-break for free);
//   * each active digit pass is a single sweep: tiles of 4096 keys are
//     ranked in shared memory (warp match + per-warp histograms, stable),
//     the per-digit tile offsets come from a decoupled look-back across
//     tiles taken in ticket order, and each tile is written out bin by bin.
// Passes that the plan marks inactive return at once, so the host never
// waits for the plan.
#include "maps_internal.cuh"

#include <algorithm>

namespace maps {
namespace {

constexpr int kRadix = 256;
constexpr int kPassThreads = 512;
constexpr int kIPT = 8;
constexpr int kTile = kPassThreads * kIPT;  // 4096 keys per tile
constexpr int kPassWarps = kPassThreads / 32;
constexpr int kLoPasses = 4;   // arrival digits
constexpr int kHiPasses = 8;   // key digits (only the low ones can vary)
constexpr int kPasses = kLoPasses + kHiPasses;
constexpr unsigned long long kAgg = 1ull << 62, kInc = 2ull << 62;
constexpr unsigned long long kValMask = 0xffffffffull;

enum : int32_t { kBufA = 0, kBufB = 1, kHiIdentity = 2, kPermOut = 2 };

struct OrderCounts {
  uint32_t h[kPasses][kRadix];
  uint32_t unsorted;
};

struct OrderPlan {
  int32_t active[kPasses];
  int32_t src[kPasses];
  int32_t dst[kPasses];
  int32_t gather_buf;  // -1: none
  int32_t npasses;
  uint32_t digit_off[kPasses][kRadix];
};

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Warp-aggregated shared-memory increment of bin `b` (all lanes active).
__device__ __forceinline__ void warp_count(uint32_t *hist, int b, bool valid) {
  const unsigned peers = __match_any_sync(0xffffffffu, valid ? b : -1);
  const int lane = threadIdx.x & 31;
  if (valid && lane == __ffs(peers) - 1) atomicAdd(&hist[b], static_cast<uint32_t>(__popc(peers)));
}

__global__ void __launch_bounds__(512)
order_prep_kernel(int64_t N, int D, int n_hi, const int32_t *__restrict__ dec,
                  const int32_t *__restrict__ bound, const int32_t *__restrict__ wait,
                  const int32_t *__restrict__ arrival, int32_t max_wait,
                  unsigned long long *hi_orig, unsigned long long *keyA, uint32_t *valA,
                  OrderCounts *counts, uint32_t *dec_count, int32_t *status) {
  __shared__ uint32_t sh[kPasses][kRadix];
  for (int i = threadIdx.x; i < kPasses * kRadix; i += blockDim.x) (&sh[0][0])[i] = 0;
  __syncthreads();
  bool bad = false, unsorted = false;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  // the loop bound depends only on the block's first index, so whole warps
  // iterate together and the warp-wide matches below see every lane
  for (int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x; i0 < N; i0 += stride) {
    const int64_t i = i0 + threadIdx.x;
    const bool valid = i < N;
    unsigned long long hi = 0;
    uint32_t a = 0;
    if (valid) {
      int32_t d = dec[i], u = bound[i], w = wait[i], ar = arrival[i];
      if (d < 0 || d >= D || u < 0 || ar < 0) {
        bad = true;
        d = d < 0 || d >= D ? 0 : d;
        u = u < 0 ? 0 : u;
        ar = ar < 0 ? 0 : ar;
      }
      const bool promoted = w > max_wait;
      const uint32_t prim = static_cast<uint32_t>(promoted ? ar : u);
      hi = (static_cast<unsigned long long>(d) << 32) |
           (static_cast<unsigned long long>(promoted ? 0u : 1u) << 31) | prim;
      a = static_cast<uint32_t>(ar);
      hi_orig[i] = hi;
      keyA[i] = a;
      valA[i] = static_cast<uint32_t>(i);
      atomicAdd(&dec_count[d], 1u);
      if (i + 1 < N && arrival[i + 1] < ar) unsorted = true;
    }
#pragma unroll
    for (int p = 0; p < kLoPasses; ++p) warp_count(sh[p], (a >> (8 * p)) & 255u, valid);
    for (int p = 0; p < n_hi; ++p)
      warp_count(sh[kLoPasses + p], static_cast<int>((hi >> (8 * p)) & 255u), valid);
  }
  if (bad) flag_error(status, MAPS_E_RANGE);
  if (__syncthreads_or(unsorted) && threadIdx.x == 0) atomicOr(&counts->unsorted, 1u);
  for (int i = threadIdx.x; i < kPasses * kRadix; i += blockDim.x) {
    const uint32_t c = (&sh[0][0])[i];
    if (c) atomicAdd(&(&counts->h[0][0])[i], c);
  }
}

// One block: digit offsets, active passes, buffer assignment, and the
// decoder segment offsets.
__global__ void __launch_bounds__(kRadix)
order_plan_kernel(int64_t N, int D, int n_hi, const OrderCounts *counts, OrderPlan *plan,
                  const uint32_t *dec_count, int64_t *seg_off) {
  __shared__ uint32_t s_warp[kRadix / 32];
  __shared__ long long s_w64[kRadix / 32];
  __shared__ int s_trivial[kPasses];
  __shared__ long long s_carry;
  const int b = threadIdx.x, lane = b & 31, warp = b >> 5;
  for (int p = 0; p < kPasses; ++p) {
    const uint32_t c = counts->h[p][b];
    uint32_t incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_warp[warp] = incl;
    const int triv = __syncthreads_or(static_cast<int64_t>(c) == N);
    uint32_t base = 0;
    for (int w = 0; w < warp; ++w) base += s_warp[w];
    plan->digit_off[p][b] = base + incl - c;
    if (b == 0) s_trivial[p] = triv;
    __syncthreads();
  }
  if (b == 0) {
    const bool unsorted = counts->unsorted != 0;
    int last = -1, n = 0, buf = kBufA;  // buffer holding the current keys
    for (int p = 0; p < kPasses; ++p) plan->active[p] = 0;
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
    s_carry = 0;
  }
  __syncthreads();
  // seg_off = exclusive scan of the per-decoder counts
  for (int base = 0; base <= D; base += kRadix) {
    const int k = base + b;
    const long long c = k < D ? dec_count[k] : 0;
    long long incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_w64[warp] = incl;
    __syncthreads();
    long long wb = 0;
    for (int w = 0; w < warp; ++w) wb += s_w64[w];
    const long long carry = s_carry;
    if (k <= D) seg_off[k] = carry + wb + incl - c;
    __syncthreads();
    if (b == kRadix - 1) s_carry = carry + wb + incl;
    __syncthreads();
  }
}

// After arrival passes: keys of the hi passes follow the arrival order.
__global__ void order_gather_kernel(int64_t N, const OrderPlan *plan, const unsigned long long *hi_orig,
                                    unsigned long long *keyA, unsigned long long *keyB,
                                    const uint32_t *valA, const uint32_t *valB) {
  const int gb = plan->gather_buf;
  if (gb < 0) return;
  unsigned long long *k = gb == kBufA ? keyA : keyB;
  const uint32_t *v = gb == kBufA ? valA : valB;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < N; i += stride)
    k[i] = hi_orig[v[i]];
}

// No active pass at all: the identity is the order.
__global__ void order_identity_kernel(int64_t N, const OrderPlan *plan, int32_t *perm) {
  if (plan->npasses != 0) return;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < N; i += stride)
    perm[i] = static_cast<int32_t>(i);
}

struct PassSmem {
  unsigned long long keys[kTile];
  uint32_t vals[kTile];
  uint32_t hw[kPassWarps][kRadix];  // per-warp counts, then per-warp bin bases
  uint32_t tile_cnt[kRadix];
  uint32_t bin_start[kRadix];       // tile-local start of each bin
  uint32_t excl[kRadix];            // global offset of this tile within each bin
  uint32_t scan_w[kRadix / 32];
  int tile;
};

__global__ void __launch_bounds__(kPassThreads)
order_pass_kernel(int p, int64_t N, const OrderPlan *plan, unsigned long long *keyA,
                  unsigned long long *keyB, uint32_t *valA, uint32_t *valB,
                  const unsigned long long *hi_orig, int32_t *perm, unsigned long long *tstatus,
                  uint32_t *ticket, int32_t *status) {
  if (!plan->active[p]) return;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  PassSmem &sm = *reinterpret_cast<PassSmem *>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int src = plan->src[p], dst = plan->dst[p];
  const int shift = p < kLoPasses ? 8 * p : 8 * (p - kLoPasses);
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
  const int64_t base = static_cast<int64_t>(tile) * kTile;

  // load and rank within the warp (stable: warp-major, then item, then lane)
  unsigned long long key[kIPT];
  uint32_t val[kIPT];
  int dig[kIPT];
  uint32_t rank[kIPT];
#pragma unroll
  for (int it = 0; it < kIPT; ++it) {
    const int64_t idx = base + warp * (32 * kIPT) + it * 32 + lane;
    const bool valid = idx < N;
    key[it] = valid ? kin[idx] : 0ull;
    val[it] = valid ? (identity ? static_cast<uint32_t>(idx) : vin[idx]) : 0u;
    dig[it] = valid ? static_cast<int>((key[it] >> shift) & 255u) : kRadix;
    const unsigned peers = __match_any_sync(0xffffffffu, dig[it]);
    const uint32_t before = __popc(peers & lanemask_lt());
    uint32_t cur = 0;
    if (valid) cur = sm.hw[warp][dig[it]];
    __syncwarp();
    if (valid && lane == __ffs(peers) - 1) sm.hw[warp][dig[it]] = cur + __popc(peers);
    __syncwarp();
    rank[it] = cur + before;
  }
  __syncthreads();
  // per bin: exclusive scan over warps, tile total
  if (tid < kRadix) {
    uint32_t run = 0;
    for (int w = 0; w < kPassWarps; ++w) {
      const uint32_t c = sm.hw[w][tid];
      sm.hw[w][tid] = run;
      run += c;
    }
    sm.tile_cnt[tid] = run;
    // publish this tile's count, then look back for the offset of the tile
    unsigned long long *st = tstatus + static_cast<size_t>(tile) * kRadix;
    if (tile == 0) {
      st_release_u64(st + tid, kInc | run);
      sm.excl[tid] = 0;
    } else {
      st_release_u64(st + tid, kAgg | run);
      unsigned long long excl = 0;
      for (int q = tile - 1; q >= 0; --q) {
        const unsigned long long *w = tstatus + static_cast<size_t>(q) * kRadix + tid;
        unsigned long long v;
        uint32_t spins = 0;
        while (((v = ld_acquire_u64(w)) >> 62) == 0) {
          if (++spins > kSpinLimit) {
            flag_error(status, MAPS_E_TIMEOUT);
            v = kInc;
            break;
          }
          __nanosleep(32);
        }
        excl += v & kValMask;
        if ((v >> 62) == 2) break;
      }
      st_release_u64(st + tid, kInc | (excl + run));
      sm.excl[tid] = static_cast<uint32_t>(excl);
    }
  }
  __syncthreads();
  // tile-local bin starts (exclusive scan of tile counts over 256 bins; the
  // first 8 warps hold the 256 bins, so every shuffle below has full warps)
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
    if (keys_out) kout[pos] = k;
    vout[pos] = sm.vals[s];
  }
}

struct OrderWs {
  OrderCounts *counts;
  uint32_t *dec_count;
  uint32_t *tickets;
  unsigned long long *tstatus;
  OrderPlan *plan;
  unsigned long long *hi_orig, *keyA, *keyB;
  uint32_t *valA, *valB;
  size_t zero_bytes;  // counts .. tstatus are contiguous and zeroed per call
};

OrderWs carve_order(Carve &c, int64_t N, int D) {
  OrderWs w;
  const int64_t tiles = (N + kTile - 1) / kTile;
  const size_t zero_begin = c.off;
  w.counts = c.take<OrderCounts>(1);
  w.dec_count = c.take<uint32_t>(static_cast<size_t>(D));
  w.tickets = c.take<uint32_t>(kPasses);
  w.tstatus = c.take<unsigned long long>(static_cast<size_t>(kPasses) * (tiles > 0 ? tiles : 1) * kRadix);
  const size_t zero_end = c.off;
  w.zero_bytes = zero_end - ((zero_begin + kAlign - 1) / kAlign * kAlign);
  w.plan = c.take<OrderPlan>(1);
  const size_t n = static_cast<size_t>(N > 0 ? N : 1);
  w.hi_orig = c.take<unsigned long long>(n);
  w.keyA = c.take<unsigned long long>(n);
  w.keyB = c.take<unsigned long long>(n);
  w.valA = c.take<uint32_t>(n);
  w.valB = c.take<uint32_t>(n);
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
  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.counts, 0, w.zero_bytes, s)));
  // key digits that can differ: bits [0, 32 + bits(D - 1))
  int dbits = 0;
  while ((1ll << dbits) < D) ++dbits;
  const int n_hi = std::min(kHiPasses, (32 + dbits + 7) / 8);
  const int sms = sm_count();
  const int64_t tiles = (N + kTile - 1) / kTile;
  if (N > 0) {
    const int gprep = static_cast<int>(std::min<int64_t>((N + 511) / 512, 2LL * sms));
    order_prep_kernel<<<gprep, 512, 0, s>>>(N, D, n_hi, dec, bound, wait, arrival, max_wait,
                                            w.hi_orig, w.keyA, w.valA, w.counts, w.dec_count, status);
  }
  order_plan_kernel<<<1, kRadix, 0, s>>>(N, D, n_hi, w.counts, w.plan, w.dec_count, seg_off_out);
  MAPS_TRY(launch_ok());
  if (N == 0) return MAPS_OK;
  const size_t smem = sizeof(PassSmem);
  MAPS_TRY(cuda_ok(cudaFuncSetAttribute(order_pass_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(smem))));
  const int gcopy = static_cast<int>(std::min<int64_t>((N + 255) / 256, 4LL * sms));
  for (int p = 0; p < kLoPasses; ++p)
    order_pass_kernel<<<static_cast<unsigned>(tiles), kPassThreads, smem, s>>>(
        p, N, w.plan, w.keyA, w.keyB, w.valA, w.valB, w.hi_orig, perm_out,
        w.tstatus + static_cast<size_t>(p) * tiles * kRadix, w.tickets + p, status);
  order_gather_kernel<<<gcopy, 256, 0, s>>>(N, w.plan, w.hi_orig, w.keyA, w.keyB, w.valA, w.valB);
  for (int p = kLoPasses; p < kLoPasses + n_hi; ++p)
    order_pass_kernel<<<static_cast<unsigned>(tiles), kPassThreads, smem, s>>>(
        p, N, w.plan, w.keyA, w.keyB, w.valA, w.valB, w.hi_orig, perm_out,
        w.tstatus + static_cast<size_t>(p) * tiles * kRadix, w.tickets + p, status);
  order_identity_kernel<<<gcopy, 256, 0, s>>>(N, w.plan, perm_out);
  return launch_ok();
}

}  // extern "C"
