// occupancy.cu -- projected KV-token occupancy over the step horizon.
//
// K[k][t] = sum over residents r of decoder k with t < e_r of (b_r + t),
// b_r = p_r + g_r + 1, e_r = min(max(U_r - g_r, 1), H), which is
//   K[k][t] = SumB_k(t) + t * Cnt_k(t)
// with Cnt / SumB the count and b-sum of residents still live at t.
//
// Layout of the work.  One CTA owns one decoder and a chunk of up to four
// horizon tiles of W steps.  It loads the decoder's residents once, keeps
// each resident's footprint at t = 0 (b) and end step (e) in shared memory,
// and walks its tiles from the highest down.  For a tile, residents ending
// inside it go into a shared-memory end-step histogram; those ending after
// it form the tile's carry (count, b-sum), which is the previous tile's carry
// plus the previous tile's bin totals.  A reverse scan of the histogram
// gives each cell's live count and b-sum, and the tile is written with
// 128-bit stores.  Chunks of the same decoder re-read the residents from L2.
// Optionally every group of 16 steps also yields
// kmax[k][t/16] = max (K[k][t] + t), a summary the dispatch uses for the
// prefix maxima of earlier horizon tiles.
//
// Integer range: every resident is live at t = 0, so K[k][0] = sum of b_r
// and every partial sum is at most K[k][0]; if that total exceeds INT32_MAX
// the call reports MAPS_E_RANGE, otherwise the 32-bit shared-memory sums
// cannot wrap and each cell is formed exactly in 64 bits.
#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kOccThreads = 512;
constexpr int kWarps = kOccThreads / 32;
constexpr int kTilesPerChunk = 2;
constexpr int kBlock = 16;    // steps per kmax summary entry
constexpr int kStage = 4096;  // residents staged in shared memory at a time

template <int CPT, bool VEC>
__global__ void __launch_bounds__(kOccThreads, 2)
occupancy_kernel(int D, int H, int TPC, int G, const int64_t *__restrict__ res_off, int64_t R,
                 const int32_t *__restrict__ prompt, const int32_t *__restrict__ gen,
                 const int32_t *__restrict__ bound, int32_t *__restrict__ K,
                 uint32_t *__restrict__ kmax, int32_t *status) {
  constexpr int W = kOccThreads * CPT;
  // Bins are padded by 4 words after every CPT bins so that the threads'
  // 16-byte reads of their own CPT bins fall on distinct banks.
  constexpr int kPad = CPT == 4 ? 0 : 4;
  constexpr int WP = W + (W / CPT) * kPad;
  __shared__ __align__(16) int32_t s_cnt[WP];  // bin j: residents whose last live step is t0 + j
  __shared__ __align__(16) int32_t s_sb[WP];   // ... and the sum of their b
  __shared__ int2 s_res[kStage];              // residents ending inside the chunk: (b, e)
  __shared__ int s_nin;                       // entries in s_res
  __shared__ long long s_red[3][kWarps];
  __shared__ uint32_t s_wsum[2][kWarps];      // per-warp bin totals, then exclusive suffixes
  __shared__ long long s_carry[2][2];         // [tile parity][count, b-sum]

  const int k = blockIdx.x / G, chunk = blockIdx.x - (blockIdx.x / G) * G;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t tile_lo = static_cast<int64_t>(chunk) * TPC;
  const int64_t tiles_all = (static_cast<int64_t>(H) + W - 1) / W;
  const int ntile = static_cast<int>(min(static_cast<int64_t>(TPC), tiles_all - tile_lo));
  const int64_t chunk_start = tile_lo * W;             // first step of this chunk
  const int64_t chunk_end = (tile_lo + ntile) * W;     // first step after it

  int64_t lo = res_off[k], hi = res_off[k + 1];
  if (lo < 0 || hi < lo || hi > R) {
    if (tid == 0 && chunk == 0) flag_error(status, MAPS_E_RANGE);
    lo = hi = 0;
  }
  const int64_t nres = hi - lo;
  bool bad = false;
  long long carry_c = 0, carry_s = 0, total_b = 0;

  // Read residents [b0, b0 + n): the ones ending inside the chunk are
  // appended to s_res (warp-aggregated), the ones live past it only add to
  // the chunk's carry; all loads of a thread are issued before use.
  constexpr int kPer = kStage / kOccThreads;
  auto gather = [&](int64_t b0, int n, bool count) {
    int32_t p[kPer], gg[kPer], U[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const int i = j * kOccThreads + tid;
      const int64_t r = lo + b0 + i;
      const bool ok = i < n;
      p[j] = ok ? __ldg(prompt + r) : 0;
      gg[j] = ok ? __ldg(gen + r) : 0;
      U[j] = ok ? __ldg(bound + r) : 0;
    }
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const int i = j * kOccThreads + tid;
      bool keep = false;
      int2 v = make_int2(0, 0);
      if (i < n) {
        if ((p[j] | gg[j] | U[j]) < 0) {
          bad = true;
        } else {
          const long long b = static_cast<long long>(p[j]) + gg[j] + 1;
          long long e = static_cast<long long>(U[j]) - gg[j];
          e = e < 1 ? 1 : (e > H ? H : e);
          if (b > 0x7fffffffLL) bad = true;  // K[k][0] = sum of b overflows
          const int32_t b32 = static_cast<int32_t>(b > 0x7fffffffLL ? 0x7fffffffLL : b);
          if (count) {
            total_b += b32;
            if (e > chunk_end) {
              carry_c += 1;
              carry_s += b32;
            }
          }
          keep = e > chunk_start && e <= chunk_end;
          v = make_int2(b32, static_cast<int32_t>(e));
        }
      }
      const unsigned m = __ballot_sync(0xffffffffu, keep);
      int base = 0;
      if (lane == 0 && m) base = atomicAdd(&s_nin, __popc(m));
      base = __shfl_sync(0xffffffffu, base, 0);
      if (keep) s_res[base + __popc(m & ((1u << lane) - 1u))] = v;
    }
  };

  // 1. Carry into the chunk's highest tile, the decoder's sum of b, and (when
  //    they fit) the chunk's own residents staged once for all its tiles.
  const bool staged_once = nres <= kStage;
  if (tid == 0) s_nin = 0;
  __syncthreads();
  for (int64_t b0 = 0; b0 < nres; b0 += kStage) {
    const int n = static_cast<int>(min(static_cast<int64_t>(kStage), nres - b0));
    gather(b0, n, true);
    if (!staged_once) {
      __syncthreads();
      if (tid == 0) s_nin = 0;  // batches are re-read per tile below
      __syncthreads();
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    carry_c += __shfl_xor_sync(0xffffffffu, carry_c, off);
    carry_s += __shfl_xor_sync(0xffffffffu, carry_s, off);
    total_b += __shfl_xor_sync(0xffffffffu, total_b, off);
  }
  if (lane == 0) {
    s_red[0][warp] = carry_c;
    s_red[1][warp] = carry_s;
    s_red[2][warp] = total_b;
  }
  for (int i = tid; i < WP; i += kOccThreads) {
    s_cnt[i] = 0;
    s_sb[i] = 0;
  }
  __syncthreads();
  if (tid == 0) {
    long long a = 0, b = 0, t = 0;
    for (int w = 0; w < kWarps; ++w) {
      a += s_red[0][w];
      b += s_red[1][w];
      t += s_red[2][w];
    }
    s_carry[(ntile - 1) & 1][0] = a;
    s_carry[(ntile - 1) & 1][1] = b;
    if (chunk == 0 && t > 0x7fffffffLL) flag_error(status, MAPS_E_RANGE);
  }

  // 2. Tiles from the highest down; tile ti reads its carry from slot ti & 1
  //    and leaves the next lower tile's in the other slot.  Histograms start
  //    zeroed; each thread
  //    clears its own bins as it reads them.
  bool over = false;
  for (int ti = ntile - 1; ti >= 0; --ti) {
    const int64_t t0 = (tile_lo + ti) * W;
    for (int64_t b0 = 0; b0 < nres; b0 += kStage) {
      if (!staged_once) {
        __syncthreads();
        if (tid == 0) s_nin = 0;
        __syncthreads();
        gather(b0, static_cast<int>(min(static_cast<int64_t>(kStage), nres - b0)), false);
      }
      __syncthreads();
      const int nin = s_nin;
      for (int i = tid; i < nin; i += kOccThreads) {
        const int2 v = s_res[i];
        const long long e = v.y;
        if (e > t0 && e <= t0 + W) {
          const int j = static_cast<int>(e - t0 - 1);  // last live cell, 0..W-1
          const int jp = j + (j / CPT) * kPad;
          atomicAdd(&s_cnt[jp], 1);
          atomicAdd(&s_sb[jp], v.x);  // exact while sum b fits int32
        }
      }
      if (staged_once) break;
    }
    __syncthreads();

    // Thread tid owns cells l = tid*CPT + c and the bins with the same index.
    // Cell l needs every bin j >= l: its own bins from l up plus all bins of
    // the threads above it.  All sums stay below K[k][0] <= INT32_MAX unless
    // a range error is already flagged, so they are kept in 32 bits.
    int32_t *cb = &s_cnt[tid * (CPT + kPad)], *sb = &s_sb[tid * (CPT + kPad)];
    uint32_t tot_c = 0, tot_s = 0;
#pragma unroll
    for (int c = 0; c < CPT; c += 4) {
      const int4 x = *reinterpret_cast<const int4 *>(cb + c);
      const int4 y = *reinterpret_cast<const int4 *>(sb + c);
      tot_c += static_cast<uint32_t>(x.x + x.y + x.z + x.w);
      tot_s += static_cast<uint32_t>(y.x + y.y + y.z + y.w);
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
      s_wsum[0][warp] = suf_c;
      s_wsum[1][warp] = suf_s;
    }
    __syncthreads();
    if (warp == 0) {  // exclusive suffix over the warps' totals
      uint32_t wc = lane < kWarps ? s_wsum[0][lane] : 0u;
      uint32_t ws = lane < kWarps ? s_wsum[1][lane] : 0u;
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
      __syncwarp();
      if (lane < kWarps) {
        s_wsum[0][lane] = wc - oc;
        s_wsum[1][lane] = ws - os;
      }
      if (lane == 0) {  // the next lower tile also carries this tile's residents
        s_red[0][0] = wc;
        s_red[1][0] = ws;
      }
    }
    __syncthreads();
    const long long cc = s_carry[ti & 1][0], cs = s_carry[ti & 1][1];
    uint32_t run_c = static_cast<uint32_t>(cc) + s_wsum[0][warp] + (suf_c - tot_c);
    uint32_t run_s = static_cast<uint32_t>(cs) + s_wsum[1][warp] + (suf_s - tot_s);

    uint32_t bmax = 0;  // max of K + t over this thread's valid cells
    const int64_t cell0 = t0 + static_cast<int64_t>(tid) * CPT;
    const uint32_t tc0 = static_cast<uint32_t>(cell0);
    int32_t *row = K + static_cast<int64_t>(k) * H;
    const bool full = cell0 + CPT <= H;
    bool ovf = false;
#pragma unroll
    for (int c0 = CPT - 4; c0 >= 0; c0 -= 4) {
      const int4 x = *reinterpret_cast<const int4 *>(cb + c0);
      const int4 y = *reinterpret_cast<const int4 *>(sb + c0);
      *reinterpret_cast<int4 *>(cb + c0) = make_int4(0, 0, 0, 0);
      *reinterpret_cast<int4 *>(sb + c0) = make_int4(0, 0, 0, 0);
      const int32_t xc[4] = {x.x, x.y, x.z, x.w}, xs[4] = {y.x, y.y, y.z, y.w};
      uint32_t o[4];
#pragma unroll
      for (int c = 3; c >= 0; --c) {
        run_c += static_cast<uint32_t>(xc[c]);
        run_s += static_cast<uint32_t>(xs[c]);
        const uint32_t t = tc0 + c0 + c;
        // K = run_s + t * run_c, exact in 64 bits
        const unsigned long long v = static_cast<unsigned long long>(t) * run_c + run_s;
        o[c] = static_cast<uint32_t>(v);
        const bool valid = full || (cell0 + c0 + c < H);
        ovf |= valid && (v >> 31) != 0;
        const uint32_t xm = valid ? o[c] + t : 0u;
        bmax = xm > bmax ? xm : bmax;
      }
      if (VEC && full) {
        *reinterpret_cast<int4 *>(row + cell0 + c0) = make_int4(o[0], o[1], o[2], o[3]);
      } else {
#pragma unroll
        for (int c = 0; c < 4; ++c)
          if (cell0 + c0 + c < H) row[cell0 + c0 + c] = static_cast<int32_t>(o[c]);
      }
    }
    over |= ovf;
    if (kmax != nullptr) {
      constexpr int L = kBlock / CPT > 0 ? kBlock / CPT : 1;  // lanes per 16-step block
#pragma unroll
      for (int off = L / 2; off > 0; off >>= 1) {
        const uint32_t y = __shfl_xor_sync(0xffffffffu, bmax, off);
        bmax = y > bmax ? y : bmax;
      }
      if ((lane % L) == 0 && cell0 < H) {
        const int64_t nb = (static_cast<int64_t>(H) + kBlock - 1) / kBlock;
        kmax[static_cast<int64_t>(k) * nb + cell0 / kBlock] = bmax;
      }
    }
    if (tid == 0) {
      s_carry[(ti & 1) ^ 1][0] = cc + s_red[0][0];
      s_carry[(ti & 1) ^ 1][1] = cs + s_red[1][0];
    }
    __syncthreads();
  }
  if (bad || over) flag_error(status, MAPS_E_RANGE);
}

int launch_occ(int cpt, bool vec, int64_t blocks, cudaStream_t s, int D, int H, int TPC, int G,
               const int64_t *res_off, int64_t R, const int32_t *prompt, const int32_t *gen,
               const int32_t *bound, int32_t *K, uint32_t *kmax, int32_t *status) {
  const dim3 grid(static_cast<unsigned>(blocks));
  if (cpt == 16) {
    if (vec)
      occupancy_kernel<16, true><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                              bound, K, kmax, status);
    else
      occupancy_kernel<16, false><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                               bound, K, kmax, status);
  } else if (cpt == 8) {
    if (vec)
      occupancy_kernel<8, true><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                             bound, K, kmax, status);
    else
      occupancy_kernel<8, false><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                              bound, K, kmax, status);
  } else if (cpt == 4) {
    if (vec)
      occupancy_kernel<4, true><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                             bound, K, kmax, status);
    else
      occupancy_kernel<4, false><<<grid, kOccThreads, 0, s>>>(D, H, TPC, G, res_off, R, prompt, gen,
                                                              bound, K, kmax, status);
  }
  return launch_ok();
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_project_occupancy_workspace_size(int32_t D, int32_t H, int64_t R) {
  (void)D;
  (void)H;
  (void)R;
  return maps::kCtrlBytes;
}

int maps_project_occupancy(int32_t D, int32_t H, const int64_t *res_off, int64_t R,
                           const int32_t *prompt, const int32_t *gen, const int32_t *bound,
                           int32_t *K_out, uint32_t *kmax_out, void *ws, size_t ws_bytes,
                           void *stream) {
  using namespace maps;
  if (D < 1 || H < 1 || R < 0 || res_off == nullptr || K_out == nullptr) return MAPS_E_INVALID;
  if (R > 0 && (prompt == nullptr || gen == nullptr || bound == nullptr)) return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_project_occupancy_workspace_size(D, H, R)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  const int cpt = H <= 2048 ? 4 : (H <= 8192 ? 8 : 16);
  const int64_t W = static_cast<int64_t>(kOccThreads) * cpt;
  const int64_t tiles = (H + W - 1) / W;
  const int TPC = static_cast<int>(tiles < kTilesPerChunk ? tiles : kTilesPerChunk);
  const int64_t G = (tiles + TPC - 1) / TPC;
  const int64_t blocks = static_cast<int64_t>(D) * G;
  if (blocks > 0x7fffffffLL) return MAPS_E_INVALID;
  const bool vec = (H % 4 == 0) && aligned(K_out, 16);
  return launch_occ(cpt, vec, blocks, s, D, H, TPC, static_cast<int>(G), res_off, R, prompt, gen,
                    bound, K_out, kmax_out, status);
}

}  // extern "C"
