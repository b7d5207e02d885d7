// occupancy.cu -- projected KV-token occupancy over the step horizon.
//
// K[k][t] = sum over residents r of decoder k with t < e_r of (b_r + t),
// b_r = p_r + g_r + 1, e_r = min(max(U_r - g_r, 1), H), which is
//   K[k][t] = SumB_k(t) + t * Cnt_k(t)
// with Cnt / SumB the count and b-sum of residents ending after t.
//
// One CTA owns one (decoder, horizon tile of W steps).  It sweeps the
// decoder's residents once: a resident ending inside the tile goes into a
// shared-memory difference histogram at its end step; one ending at or after
// the tile's end only adds to the carry (count, b-sum) that every cell of the
// tile sees.  The carry is therefore computed directly by each tile and no
// tile waits on another.  A reverse scan of the histogram then gives each
// cell's suffix count and sum, and the tile is written with 128-bit stores.
//
// Integer range: every resident is live at t = 0, so K[k][0] = sum of b_r
// over the decoder and every partial sum in the tile is at most K[k][0].  If
// that total exceeds INT32_MAX the call reports MAPS_E_RANGE; otherwise the
// 32-bit shared-memory sums cannot wrap and each cell is formed exactly in
// 64 bits before its own range check.
#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kOccThreads = 512;
constexpr int kWarps = kOccThreads / 32;

template <int CPT, bool VEC>
__global__ void __launch_bounds__(kOccThreads)
occupancy_kernel(int D, int H, int T, const int64_t *__restrict__ res_off, int64_t R,
                 const int32_t *__restrict__ prompt, const int32_t *__restrict__ gen,
                 const int32_t *__restrict__ bound, int32_t *__restrict__ K, int32_t *status) {
  constexpr int W = kOccThreads * CPT;
  __shared__ int32_t s_cnt[W + 1];  // bin m (1..W-1): residents ending at t0 + m
  __shared__ int32_t s_sb[W + 1];   // ... and the sum of their b
  __shared__ long long s_red[3][kWarps];
  __shared__ int32_t s_scan[2][kWarps];

  const int k = blockIdx.x / T;
  const int tile = blockIdx.x - k * T;
  const int64_t t0 = static_cast<int64_t>(tile) * W;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  for (int i = tid; i <= W; i += kOccThreads) {
    s_cnt[i] = 0;
    s_sb[i] = 0;
  }
  int64_t lo = res_off[k], hi = res_off[k + 1];
  if (lo < 0 || hi < lo || hi > R) {
    if (tid == 0) flag_error(status, MAPS_E_RANGE);
    lo = hi = 0;
  }
  __syncthreads();

  long long carry_c = 0, carry_s = 0, total_b = 0;
  bool bad = false;
  for (int64_t r = lo + tid; r < hi; r += kOccThreads) {
    const int32_t p = __ldg(prompt + r), g = __ldg(gen + r), U = __ldg(bound + r);
    if ((p | g | U) < 0) {
      bad = true;
      continue;
    }
    const long long b = static_cast<long long>(p) + g + 1;
    long long e = static_cast<long long>(U) - g;
    e = e < 1 ? 1 : (e > H ? H : e);
    total_b += b;
    if (e >= t0 + W) {
      carry_c += 1;
      carry_s += b;
    } else if (e > t0) {
      const int m = static_cast<int>(e - t0);
      atomicAdd(&s_cnt[m], 1);
      atomicAdd(&s_sb[m], static_cast<int32_t>(b));  // exact when total_b fits int32
    }
  }
  if (bad) flag_error(status, MAPS_E_RANGE);

  // block sums of the carry and of the decoder's total b
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
  __syncthreads();
  carry_c = carry_s = total_b = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    carry_c += s_red[0][w];
    carry_s += s_red[1][w];
    total_b += s_red[2][w];
  }
  if (total_b > 0x7fffffffLL && tid == 0 && tile == 0) flag_error(status, MAPS_E_RANGE);

  // Thread tid owns cells l = tid*CPT + c and bins m = l + 1.  Cell l needs
  // the sums over bins m > l: its own bins above l plus every bin of the
  // threads above it (an exclusive suffix scan of the per-thread totals).
  int32_t own_c[CPT], own_s[CPT];
  int32_t tot_c = 0, tot_s = 0;
#pragma unroll
  for (int c = 0; c < CPT; ++c) {
    own_c[c] = s_cnt[tid * CPT + c + 1];
    own_s[c] = s_sb[tid * CPT + c + 1];
    tot_c += own_c[c];
    tot_s += own_s[c];
  }
  int32_t suf_c = tot_c, suf_s = tot_s;  // inclusive suffix within the warp
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int32_t yc = __shfl_down_sync(0xffffffffu, suf_c, off);
    const int32_t ys = __shfl_down_sync(0xffffffffu, suf_s, off);
    if (lane + off < 32) {
      suf_c += yc;
      suf_s += ys;
    }
  }
  if (lane == 0) {
    s_scan[0][warp] = suf_c;
    s_scan[1][warp] = suf_s;
  }
  __syncthreads();
  long long run_c = carry_c + (suf_c - tot_c);
  long long run_s = carry_s + (suf_s - tot_s);
  for (int w = warp + 1; w < kWarps; ++w) {
    run_c += s_scan[0][w];
    run_s += s_scan[1][w];
  }

  int32_t out[CPT];
  bool over = false;
#pragma unroll
  for (int c = CPT - 1; c >= 0; --c) {
    run_c += own_c[c];
    run_s += own_s[c];
    const long long t = t0 + tid * CPT + c;
    long long v = run_s + t * run_c;
    if (v > 0x7fffffffLL) {
      if (t < H) over = true;  // only cells inside the horizon count
      v = 0x7fffffffLL;
    }
    out[c] = static_cast<int32_t>(v);
  }

  const int64_t cell0 = t0 + static_cast<int64_t>(tid) * CPT;
  int32_t *row = K + static_cast<int64_t>(k) * H;
  if (VEC) {
    // H % 4 == 0 and CPT % 4 == 0: each group of 4 is wholly inside or outside
#pragma unroll
    for (int c = 0; c < CPT; c += 4) {
      if (cell0 + c < H) {
        *reinterpret_cast<int4 *>(row + cell0 + c) = make_int4(out[c], out[c + 1], out[c + 2], out[c + 3]);
      }
    }
  } else {
#pragma unroll
    for (int c = 0; c < CPT; ++c)
      if (cell0 + c < H) row[cell0 + c] = out[c];
  }
  if (over) flag_error(status, MAPS_E_RANGE);
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
                           int32_t *K_out, void *ws, size_t ws_bytes, void *stream) {
  using namespace maps;
  if (D < 1 || H < 1 || R < 0 || res_off == nullptr || K_out == nullptr) return MAPS_E_INVALID;
  if (R > 0 && (prompt == nullptr || gen == nullptr || bound == nullptr)) return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_project_occupancy_workspace_size(D, H, R)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  const bool big = H > 512;
  const int W = kOccThreads * (big ? 8 : 1);
  const int64_t T = (static_cast<int64_t>(H) + W - 1) / W;
  const int64_t blocks = T * D;
  if (blocks > 0x7fffffffLL) return MAPS_E_INVALID;
  const bool vec = (H % 4 == 0) && aligned(K_out, 16);
  const dim3 grid(static_cast<unsigned>(blocks));
  const int Ti = static_cast<int>(T);
  if (big) {
    if (vec)
      occupancy_kernel<8, true><<<grid, kOccThreads, 0, s>>>(D, H, Ti, res_off, R, prompt, gen, bound, K_out, status);
    else
      occupancy_kernel<8, false><<<grid, kOccThreads, 0, s>>>(D, H, Ti, res_off, R, prompt, gen, bound, K_out, status);
  } else {
    occupancy_kernel<1, false><<<grid, kOccThreads, 0, s>>>(D, H, Ti, res_off, R, prompt, gen, bound, K_out, status);
  }
  return launch_ok();
}

}  // extern "C"
