// rr_pressure.cu -- the round-robin KV-pressure simulation of App. A and its
// high-pressure (HP) interval metrics, for many workload realisations at once.
//
// Model (App. A): requests arrive in order; round robin sends request i to
// decoder i mod N (App. A, routing equation); a request holds
// M = L_p + L_out KV tokens while admitted (Eq. kv_demand); a decoder admits
// the head of its FIFO queue while K + M(head) <= C (Eq. admission); service
// is processor sharing at one token per t_tok, taken at token granularity: a
// round gives each of the n admitted requests one token and lasts n * t_tok,
// completions and admissions happen at round boundaries (completions first),
// and an idle decoder admits a request when it arrives.  A decoder is under
// high pressure while K * 1e6 >= theta_ppm * C (Definition of the HP
// interval).  All times are integer microseconds.
//
// Under round robin the decoders never interact, so every (realisation,
// decoder) stream is simulated by one warp on its own.  The warp does not
// step round by round: between two events every admitted request gains the
// same number of tokens, so it jumps straight to the next one -- the first
// completion (the smallest finishing round among the admitted requests), or,
// when the queue is empty, the round boundary at or after the next arrival.
// The admitted requests (stream position, finishing round, footprint) live in
// the warp's shared memory; the stream's next 32 requests sit in the warp's
// registers, one per lane.  After the run the warp derives the waiting
// statistics from the admission times.  A second, small kernel turns each
// realisation's last completion into its simulated span T_sim.
#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kRRWarps = 2;      // streams per CTA
constexpr int kRunCap = 1536;    // requests one decoder may run at once
constexpr int kStats = 6;        // T_hp, B_hp, C_hp, completed, longest queue, total wait

struct RRStream {
  int32_t pos[kRunCap];  // stream position of each admitted request
  int32_t fin[kRunCap];  // the round at whose end it completes
  int32_t m[kRunCap];    // its footprint
};

__device__ __forceinline__ int64_t warp_min64(int64_t v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const int64_t y = __shfl_xor_sync(0xffffffffu, v, off);
    v = y < v ? y : v;
  }
  return v;
}
__device__ __forceinline__ int64_t warp_sum64(int64_t v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__global__ void __launch_bounds__(32 * kRRWarps)
rr_stream_kernel(int64_t n_real, int64_t n, int N, int64_t C, int64_t tok, uint32_t theta_ppm,
                 const int64_t *__restrict__ arrival, const int32_t *__restrict__ prompt,
                 const int32_t *__restrict__ out_len, int64_t *__restrict__ admit,
                 int64_t *__restrict__ done, int64_t *__restrict__ stats,
                 int64_t *__restrict__ last_done, int32_t *status) {
  pdl_prologue();
  __shared__ RRStream sm[kRRWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t stream = static_cast<int64_t>(blockIdx.x) * kRRWarps + warp;
  if (stream >= n_real * N) return;
  RRStream &rs = sm[warp];
  const int64_t r = stream / N;
  const int d = static_cast<int>(stream - r * N);
  const int64_t *A = arrival + r * n;
  const int32_t *P = prompt + r * n, *O = out_len + r * n;
  int64_t *adm = admit + r * n, *dn = done + r * n;
  int64_t *st = stats + stream * kStats;
  const int64_t n_d = d < n ? (n - 1 - d) / N + 1 : 0;  // requests d, d + N, ...

  // the stream's requests in the domain (a footprint above C would block its
  // queue for ever), and arrival in order
  bool bad = false;
  for (int64_t s = lane; s < n_d; s += 32) {
    const int64_t i = d + s * N;
    const int32_t p = P[i], o = O[i];
    if (p < 0 || o < 1 || static_cast<int64_t>(p) + o > C || A[i] < 0 || (i > 0 && A[i] < A[i - 1]))
      bad = true;
  }
  if (__any_sync(0xffffffffu, bad)) {
    if (lane == 0) {
      flag_error(status, MAPS_E_RANGE);
      for (int q = 0; q < kStats; ++q) st[q] = 0;
      last_done[stream] = 0;
    }
    return;
  }

  // window of the next 32 requests, lane j = stream position wb + j
  int64_t wb = 0, wa = 0;
  int32_t wm = 0, wo = 0;
  auto load_window = [&](int64_t base) {
    wb = base;
    const int64_t s = base + lane;
    if (s < n_d) {
      const int64_t i = d + s * N;
      wa = A[i];
      wo = O[i];
      wm = P[i] + wo;
    }
  };
  load_window(0);

  int64_t t = n_d > 0 ? A[d] : 0, R = 0, K = 0, qh = 0, completed = 0, t_last = 0;
  int n_run = 0;
  bool in_hp = false;
  int64_t t_s = 0, T_hp = 0, B_hp = 0, C_hp = 0;
  bool fail = false;
  // every iteration admits, completes, or reaches an arrival's round boundary
  const int64_t max_iter = 4 * n_d + 16;
  for (int64_t iter = 0; iter < max_iter; ++iter) {
    // admissions at t: the FIFO head while it has arrived and fits
    int64_t ha = 0;
    for (;;) {
      if (qh >= n_d) break;
      if (qh - wb >= 32) load_window(qh);
      const int src = static_cast<int>(qh - wb);
      ha = __shfl_sync(0xffffffffu, wa, src);
      const int32_t hm = __shfl_sync(0xffffffffu, wm, src);
      const int32_t ho = __shfl_sync(0xffffffffu, wo, src);
      if (ha > t || K + hm > C) break;
      if (n_run >= kRunCap || R + ho > 0x7fffffffLL) {
        fail = true;
        break;
      }
      if (lane == 0) {
        rs.pos[n_run] = static_cast<int32_t>(qh);
        rs.fin[n_run] = static_cast<int32_t>(R + ho);
        rs.m[n_run] = hm;
        adm[d + qh * N] = t;
      }
      ++n_run;
      K += hm;
      ++qh;
    }
    if (fail) break;
    // high-pressure state after every change at t
    const bool now = K * 1000000 >= static_cast<int64_t>(theta_ppm) * C;
    if (now && !in_hp) {
      in_hp = true;
      t_s = t;
    } else if (!now && in_hp) {
      in_hp = false;
      const int64_t len = t - t_s;
      T_hp += len;
      B_hp = len > B_hp ? len : B_hp;
      C_hp += 1;
    }
    if (n_run == 0) {
      if (qh >= n_d) break;
      t = ha;  // idle until the head arrives (it fits an empty decoder)
      continue;
    }
    __syncwarp();
    // next event: the first completion, or the boundary where the head arrives
    int64_t f = 0x7fffffffffffffffLL;
    for (int j = lane; j < n_run; j += 32) f = rs.fin[j] < f ? rs.fin[j] : f;
    const int64_t f_min = warp_min64(f);
    int64_t k = f_min - R;
    const int64_t step = static_cast<int64_t>(n_run) * tok;
    if (qh < n_d && ha > t) {
      const int64_t ka = (ha - t + step - 1) / step;
      k = ka < k ? ka : k;
    }
    t += k * step;
    R += k;
    if (R == f_min) {
      // completions: record them and compact the rest in place (a chunk is
      // read whole before it is written, and writes never pass the reads)
      int wpos = 0, gone = 0;
      int64_t freed = 0;
      for (int base = 0; base < n_run; base += 32) {
        const int j = base + lane;
        const bool live = j < n_run;
        const int32_t pj = live ? rs.pos[j] : 0, fj = live ? rs.fin[j] : 0, mj = live ? rs.m[j] : 0;
        const bool fin_now = live && fj == R;
        if (fin_now) {
          dn[d + static_cast<int64_t>(pj) * N] = t;
          freed += mj;
        }
        const unsigned keep = __ballot_sync(0xffffffffu, live && !fin_now);
        __syncwarp();
        if (live && !fin_now) {
          const int to = wpos + __popc(keep & ((1u << lane) - 1u));
          rs.pos[to] = pj;
          rs.fin[to] = fj;
          rs.m[to] = mj;
        }
        __syncwarp();
        wpos += __popc(keep);
        gone += __popc(__ballot_sync(0xffffffffu, fin_now));
      }
      n_run = wpos;
      K -= warp_sum64(freed);
      completed += gone;
      t_last = t;
    }
  }
  if (fail || n_run != 0 || qh < n_d) {  // capacity of the running set, or no progress
    if (lane == 0) flag_error(status, MAPS_E_RANGE);
  }
  __syncwarp();

  // waiting statistics from the admission times (non-decreasing along the
  // stream: FIFO): the total wait, and at each arrival the requests that had
  // arrived and were not yet admitted
  int64_t wait = 0, qmax = 0;
  for (int64_t s = lane; s < n_d; s += 32) {
    const int64_t i = d + s * N;
    const int64_t ai = A[i];
    wait += adm[i] - ai;
    // first position j <= s with admit_j > a_i
    int64_t lo = 0, hi = s + 1;
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (adm[d + mid * N] > ai)
        hi = mid;
      else
        lo = mid + 1;
    }
    const int64_t q = s + 1 - lo;
    qmax = q > qmax ? q : qmax;
  }
  wait = warp_sum64(wait);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const int64_t y = __shfl_xor_sync(0xffffffffu, qmax, off);
    qmax = y > qmax ? y : qmax;
  }
  if (lane == 0) {
    st[0] = T_hp;
    st[1] = B_hp;
    st[2] = C_hp;
    st[3] = completed;
    st[4] = qmax;
    st[5] = wait;
    last_done[stream] = t_last;
  }
}

// T_sim of every realisation: its last completion minus its first arrival.
__global__ void __launch_bounds__(256)
rr_span_kernel(int64_t n_real, int64_t n, int N, const int64_t *__restrict__ arrival,
               const int64_t *__restrict__ last_done, int64_t *__restrict__ t_sim) {
  pdl_prologue();
  const int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (r >= n_real) return;
  int64_t m = 0;
  for (int d = 0; d < N; ++d) m = last_done[r * N + d] > m ? last_done[r * N + d] : m;
  t_sim[r] = m - arrival[r * n];
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_rr_pressure_workspace_size(const maps_rr_cfg *cfg, int64_t n_real) {
  using namespace maps;
  Carve c(nullptr);
  if (cfg != nullptr && n_real > 0 && cfg->N > 0) c.take<int64_t>(static_cast<size_t>(n_real) * cfg->N);
  return c.bytes();
}

int maps_rr_pressure(const maps_rr_cfg *cfg, int64_t n_real, const int64_t *arrival_us,
                     const int32_t *prompt, const int32_t *out_len, int64_t *admit_us,
                     int64_t *done_us, int64_t *stats_out, int64_t *t_sim_out, void *ws,
                     size_t ws_bytes, void *stream) {
  using namespace maps;
  if (cfg == nullptr || n_real < 1 || cfg->n_req < 1 || cfg->N < 1 || cfg->C < 1 ||
      cfg->t_tok_us < 1 || cfg->theta_ppm == 0 || cfg->theta_ppm > 1000000u)
    return MAPS_E_INVALID;
  if (n_real > (int64_t(1) << 40) / cfg->n_req || n_real * cfg->N > 0x7fffffffLL * kRRWarps)
    return MAPS_E_INVALID;
  if (arrival_us == nullptr || prompt == nullptr || out_len == nullptr || admit_us == nullptr ||
      done_us == nullptr || stats_out == nullptr || t_sim_out == nullptr)
    return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_rr_pressure_workspace_size(cfg, n_real)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  Carve c(ws);
  int64_t *last = c.take<int64_t>(static_cast<size_t>(n_real) * cfg->N);
  const int64_t streams = n_real * cfg->N;
  launch_pdl(rr_stream_kernel, static_cast<unsigned>((streams + kRRWarps - 1) / kRRWarps),
             32 * kRRWarps, 0, s, n_real, cfg->n_req, cfg->N, static_cast<int64_t>(cfg->C),
             static_cast<int64_t>(cfg->t_tok_us), cfg->theta_ppm, arrival_us, prompt, out_len,
             admit_us, done_us, stats_out, last, status);
  launch_pdl(rr_span_kernel, static_cast<unsigned>((n_real + 255) / 256), 256, 0, s, n_real,
             cfg->n_req, cfg->N, arrival_us, last, t_sim_out);
  return launch_ok();
}

}  // extern "C"
