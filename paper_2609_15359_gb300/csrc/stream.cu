// stream.cu -- the streaming scheduler loop (Sec. 3.2 sliding calibration
// window, Sec. 3.3 dispatch and local order, Algorithm 1's round-robin
// fallback, App. A Eq. admission) with all state resident on the device.
//
// Per batch of arrivals, in the paper's order:
//   1. advance every running request by the steps since the last batch; a
//      request completes on reaching its true length      (stream_advance)
//   2. completions enter the calibration window in (completion step, id)
//      order: maps_order_local sorts them, stream_window writes the ring
//   3. calibrate on the window and bound every request in the system and the
//      batch (maps_calibrate); an unbounded quantile sends the batch round
//      robin                                                (stream_rr)
//   4. group running and waiting requests by decoder      (stream_csr)
//   5. dispatch the batch SEQUENTIALly with Q = the waiting counts: a walk
//      over each decoder's sorted end steps in shared memory (stream_dispatch),
//      or, where those lists do not fit, maps_project_occupancy and
//      maps_dispatch
//   6. the batch joins its decoders' waiting queues        (stream_enqueue)
//   7. local order of every waiting queue (stream_waitlist, maps_order_local)
//   8. admission in queue order while used + p + U <= capacity, the first
//      misfit blocking its queue                            (stream_admit)
// Policy variants replace step 5 (max-headroom, round-robin or least-requests
// dispatch: stream_dispatch with mc, stream_rr, stream_lr), the order of step 7
// (FCFS: every entry promoted, so arrival order alone) and what a running
// request counts for in step 8 (occupancy, staged or held reservation).
// Fidelity modes: per-step admission with preemption replaces step 1 by a
// step-by-step simulation of each decoder (stream_interval); deferral splits
// the arrived requests at each dispatch step into those with a bound, those
// timed out to round robin and those that keep waiting (stream_select).
// The host issues the launches; it reads 40 bytes of loop state once per
// batch (the request, completion and waiting counts, and the deferral's list
// lengths, that size the calls).
#include <algorithm>
#include <climits>

#include "maps_internal.cuh"

namespace maps {
namespace {

constexpr int kSt = 1024;  // threads of the one-block kernels
constexpr int kStWarps = kSt / 32;
constexpr int kStreamMaxD = 1024;
enum : uint8_t { kNotYet = 0, kWaiting = 1, kRunning = 2, kDone = 3 };

struct StreamState {
  long long prev_s;  // dispatch step of the previous batch
  int32_t nact;      // requests in the system (waiting or running)
  int32_t ndone;     // completions found by the last advance
  int32_t nwait;     // waiting requests after the last advance
  int32_t npend;     // deferral: arrived requests not yet dispatched
  int32_t nc;        // deferral: requests for the dispatch policy at this step
  int32_t nto;       // deferral: requests timed out to round robin at this step
  int32_t adm_i;     // per-step mode: admissions between the dispatch steps
  int32_t pad;
};

// Exclusive position of a 0/1 flag across the block (kSt threads) and the
// block's total.  Every thread must call it.
__device__ __forceinline__ int block_flag_scan(bool f, int *s_w, int &total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned m = __ballot_sync(0xffffffffu, f);
  if (lane == 0) s_w[warp] = __popc(m);
  __syncthreads();
  int base = 0, tot = 0;
#pragma unroll 8
  for (int w = 0; w < kStWarps; ++w) {
    const int c = s_w[w];
    base += w < warp ? c : 0;
    tot += c;
  }
  __syncthreads();
  total = tot;
  return base + __popc(m & ((1u << lane) - 1u));
}

__global__ void stream_validate_kernel(int64_t N, const int64_t *arrival, const int32_t *prompt,
                                       const int32_t *true_len, const int32_t *pred,
                                       const int32_t *pred_delay, int32_t *status) {
  pdl_prologue();
  bool bad = false;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < N; i += stride)
    if (prompt[i] < 0 || true_len[i] < 1 || pred[i] < 0 || (i > 0 && arrival[i] < arrival[i - 1]) ||
        (pred_delay != nullptr && pred_delay[i] < 0))
      bad = true;
  if (bad) flag_error(status, MAPS_E_RANGE);
}

__global__ void stream_init_kernel(int64_t first_hi, int D, int32_t cap, const int64_t *arrival,
                                   int32_t *capv, StreamState *S) {
  pdl_prologue();
  for (int k = threadIdx.x; k < D; k += blockDim.x) capv[k] = cap;
  if (threadIdx.x == 0) {
    S->prev_s = arrival[first_hi - 1];
    S->nact = 0;
    S->ndone = 0;
    S->nwait = 0;
    S->npend = 0;
    S->nc = 0;
    S->nto = 0;
    S->adm_i = 0;
  }
}

// 1. Advance by delta = s - prev_s steps; keep the survivors in id order.
//    occupancy = p + g of the running requests (the over-capacity count);
//    used = what admission counts for them: p + g, p + max(U*, g) (staged)
//    or 2p + max(U*, g) (held), U* the bound reserved at admission.
__global__ void __launch_bounds__(kSt, 1)
stream_advance_kernel(int64_t hi, int D, int32_t cap, int acct, int per_step, const int64_t *arrival,
                      const int32_t *prompt, const int32_t *true_len, const int32_t *res_u,
                      uint8_t *st, int32_t *g, const int32_t *dec, const int32_t *act_in,
                      int32_t *act_out, int32_t *done_id, int32_t *done_rem, long long *used,
                      StreamState *S, int64_t *stats_b, int64_t *dst) {
  pdl_prologue();
  __shared__ unsigned long long s_occ[kStreamMaxD], s_used[kStreamMaxD];
  __shared__ int s_w[kStWarps];
  __shared__ int s_nwait;
  const int tid = threadIdx.x;
  for (int k = tid; k < D; k += kSt) s_occ[k] = s_used[k] = 0;
  if (tid == 0) s_nwait = 0;
  const long long s = arrival[hi - 1];
  const long long delta = s - S->prev_s;  // 0 after the per-step interval
  const int nact = S->nact;
  // per-step mode: the interval kernel's completions come first
  int nkeep = 0, ndone = per_step ? S->ndone : 0, nwait = 0;
  __syncthreads();
  for (int c0 = 0; c0 < nact; c0 += kSt) {
    const int x = c0 + tid;
    int id = -1, rem32 = 0;
    bool done = false, gone = false;
    if (x < nact) {
      id = act_in[x];
      const uint8_t sv = st[id];
      gone = sv == kDone;  // completed in the per-step interval
      if (sv == kRunning) {
        const long long rem = static_cast<long long>(true_len[id]) - g[id];  // >= 1
        if (rem <= delta) {
          done = true;
          rem32 = static_cast<int>(rem);
          st[id] = kDone;
        } else {
          const int gn = g[id] + static_cast<int>(delta);  // < true_len
          g[id] = gn;
          const long long p = prompt[id];
          atomicAdd(&s_occ[dec[id]], static_cast<unsigned long long>(p + gn));
          if (acct != MAPS_STREAM_OCCUPANCY) {
            const long long out = max(static_cast<long long>(res_u[id]), static_cast<long long>(gn));
            atomicAdd(&s_used[dec[id]], static_cast<unsigned long long>(
                                            (acct == MAPS_STREAM_HELD ? 2 * p : p) + out));
          }
        }
      } else if (sv == kWaiting) {
        ++nwait;
      }
    }
    int tk, td;
    const int pk = block_flag_scan(id >= 0 && !done && !gone, s_w, tk);
    const int pd = block_flag_scan(done, s_w, td);
    if (id >= 0 && !done && !gone) act_out[nkeep + pk] = id;
    if (done) {
      done_id[ndone + pd] = id;
      done_rem[ndone + pd] = rem32;
    }
    nkeep += tk;
    ndone += td;
  }
  if (nwait) atomicAdd(&s_nwait, nwait);
  const bool ov = tid < D && static_cast<long long>(s_occ[tid]) > cap;  // D <= kSt
  if (tid < D) {
    used[tid] = static_cast<long long>(acct == MAPS_STREAM_OCCUPANCY ? s_occ[tid] : s_used[tid]);
    if (dst != nullptr && ov) dst[4 * tid + 1] += 1;
  }
  const int over = __syncthreads_count(ov);
  if (tid == 0) {
    S->prev_s = s;
    S->nact = nkeep;
    S->ndone = ndone;
    S->nwait = s_nwait;
    stats_b[0] = ndone;
    stats_b[3] = over;
  }
}

// 1'. Per-step mode: the steps prev_s + 1 .. s, one warp per decoder
//     (decoders do not interact between dispatch steps).  Each decoder holds
//     its running requests (in rbuf, unordered; the admission order is aseq)
//     and the requests it preempted since the last dispatch step (sbuf, a
//     stack, the latest on top); its waiting queue is the order computed at
//     the last dispatch step past the requests admitted then.  A step: while
//     the running requests would pass the capacity by taking one token each,
//     the most recently admitted one (never the last) is preempted, losing
//     its tokens; each takes a token, and those reaching their true length
//     complete; then, except on the dispatch step s, the stack top or the
//     queue head is admitted while used + p + U <= capacity.  Between events
//     nothing but the growth happens: no admission can succeed (used only
//     grows and nothing is freed since the head last failed), so the warp
//     jumps to the next step with a completion or a preemption, or to s.
//     Every iteration advances the step, so the loop ends.
__global__ void __launch_bounds__(kSt, 1)
stream_interval_kernel(int64_t hi, int D, int32_t cap, int acct, const int64_t *arrival,
                       const int32_t *prompt, const int32_t *true_len, const int32_t *U,
                       int32_t *res_u, uint8_t *st, int32_t *g, const int32_t *dec,
                       const int32_t *act, const int32_t *wid, const int32_t *wperm,
                       const int64_t *wseg, const int64_t *qhead, long long *aseq,
                       long long *dseq, int32_t *rbuf, int32_t *sbuf, int32_t *done_id,
                       int32_t *done_rem, StreamState *S, int64_t *dst) {
  pdl_prologue();
  __shared__ int s_cnt[kStreamMaxD], s_run[kStreamMaxD], s_cur[kStreamMaxD];
  __shared__ int s_w[kStWarps];
  __shared__ int s_done, s_adm;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const long long s = arrival[hi - 1];
  const long long s0 = S->prev_s;
  const int nact = S->nact;
  for (int k = tid; k < D; k += kSt) s_cnt[k] = s_run[k] = 0;
  if (tid == 0) s_done = s_adm = 0;
  __syncthreads();
  // each decoder's region: room for all its requests in the system
  for (int x = tid; x < nact; x += kSt) {
    const int id = act[x];
    atomicAdd(&s_cnt[dec[id]], 1);
    if (st[id] == kRunning) atomicAdd(&s_run[dec[id]], 1);
  }
  __syncthreads();
  {
    const int c = tid < D ? s_cnt[tid] : 0;  // D <= kSt
    int incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    if (lane == 31) s_w[warp] = incl;
    __syncthreads();
    int base = 0;
    for (int w = 0; w < warp; ++w) base += s_w[w];
    if (tid < D) {
      s_cnt[tid] = base + incl - c;  // now the region's start
      s_cur[tid] = 0;
    }
  }
  __syncthreads();
  for (int x = tid; x < nact; x += kSt) {
    const int id = act[x];
    if (st[id] == kRunning) {
      const int k = dec[id];
      rbuf[s_cnt[k] + atomicAdd(&s_cur[k], 1)] = id;
    }
  }
  __syncthreads();
  for (int k = warp; k < D; k += kStWarps) {
    const int base = s_cnt[k];
    int n = s_run[k], ns = 0;
    long long qh = qhead[k];
    const long long qe = wseg[k + 1];
    long long seq = dseq[k], integ = 0;
    int npre = 0, nadm = 0;
    long long t = s0;
    while (t < s) {
      long long tok = 0;
      int jc = INT_MAX;
      for (int i = lane; i < n; i += 32) {
        const int id = rbuf[base + i];
        const int gi = g[id];
        tok += static_cast<long long>(prompt[id]) + gi;
        jc = min(jc, true_len[id] - gi);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        tok += __shfl_xor_sync(0xffffffffu, tok, off);
        jc = min(jc, __shfl_xor_sync(0xffffffffu, jc, off));
      }
      // steps to the next completion (jc) and to the next preemption (jp)
      long long je = LLONG_MAX;
      if (n > 0) {
        je = jc;
        if (n > 1) je = min(je, tok + n > cap ? 1LL : (cap - tok) / n + 1);
      }
      const long long te = je >= s - t ? s : t + je;
      const long long quiet = te - t - 1;  // steps of growth alone
      if (quiet > 0) {
        for (int i = lane; i < n; i += 32) g[rbuf[base + i]] += static_cast<int>(quiet);
        integ += (static_cast<long long>(ns) + (qe - qh)) * quiet;
        tok += static_cast<long long>(n) * quiet;
      }
      t = te;
      __syncwarp();
      // step t: preempt the latest admitted while the next tokens do not fit
      while (n > 1 && tok + n > cap) {
        long long best = -1;
        int bi = 0;
        for (int i = lane; i < n; i += 32) {
          const long long a = aseq[rbuf[base + i]];
          if (a > best) {
            best = a;
            bi = i;
          }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const long long ob = __shfl_xor_sync(0xffffffffu, best, off);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
          if (ob > best) {
            best = ob;
            bi = oi;
          }
        }
        const int v = rbuf[base + bi];
        tok -= static_cast<long long>(prompt[v]) + g[v];
        __syncwarp();
        if (lane == 0) {
          rbuf[base + bi] = rbuf[base + n - 1];
          sbuf[base + ns] = v;
          st[v] = kWaiting;
          g[v] = 0;
        }
        --n;
        ++ns;
        ++npre;
        __syncwarp();
      }
      // one token each; completions leave the running set (in-place compaction)
      int kept = 0;
      for (int r0 = 0; r0 < n; r0 += 32) {
        const int i = r0 + lane;
        const int id = i < n ? rbuf[base + i] : -1;
        bool fin = false;
        if (id >= 0) {
          const int gi = g[id] + 1;
          g[id] = gi;
          fin = gi == true_len[id];
          if (fin) {
            st[id] = kDone;
            const int o = atomicAdd(&s_done, 1);
            done_id[o] = id;
            done_rem[o] = static_cast<int>(t - s0);
          }
        }
        const unsigned km = __ballot_sync(0xffffffffu, id >= 0 && !fin);
        if (id >= 0 && !fin) rbuf[base + kept + __popc(km & ((1u << lane) - 1u))] = id;
        kept += __popc(km);
        __syncwarp();
      }
      n = kept;
      if (t == s) break;
      // admission in queue order (the stack first)
      long long used = 0;
      for (int i = lane; i < n; i += 32) {
        const int id = rbuf[base + i];
        const long long p = prompt[id], gi = g[id];
        const long long out = max(static_cast<long long>(res_u[id]), gi);
        used += acct == MAPS_STREAM_OCCUPANCY ? p + gi
                : acct == MAPS_STREAM_STAGED  ? p + out
                                              : 2 * p + out;
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) used += __shfl_xor_sync(0xffffffffu, used, off);
      if (lane == 0) {
        for (;;) {
          const bool from_stack = ns > 0;
          if (!from_stack && qh >= qe) break;
          const int c = from_stack ? sbuf[base + ns - 1] : wid[wperm[qh]];
          const long long p = prompt[c], uu = U[c];
          if (used + p + uu > cap) break;
          if (from_stack)
            --ns;
          else
            ++qh;
          rbuf[base + n] = c;
          ++n;
          st[c] = kRunning;
          g[c] = 0;
          res_u[c] = static_cast<int32_t>(uu);
          aseq[c] = seq++;
          used += acct == MAPS_STREAM_OCCUPANCY ? p : acct == MAPS_STREAM_STAGED ? p + uu : 2 * p + uu;
          ++nadm;
        }
      }
      n = __shfl_sync(0xffffffffu, n, 0);
      ns = __shfl_sync(0xffffffffu, ns, 0);
      qh = __shfl_sync(0xffffffffu, qh, 0);
      seq = __shfl_sync(0xffffffffu, seq, 0);
      __syncwarp();
      integ += static_cast<long long>(ns) + (qe - qh);  // waiting through step t
    }
    if (lane == 0) {
      dseq[k] = seq;
      if (dst != nullptr) {
        dst[4 * k] += integ;
        dst[4 * k + 2] += nadm;
        dst[4 * k + 3] += npre;
      }
      if (nadm) atomicAdd(&s_adm, nadm);
    }
  }
  __syncthreads();
  if (tid == 0) {
    S->ndone = s_done;
    S->adm_i = s_adm;
    S->prev_s = s;  // the advance that follows moves nobody
  }
}

// Deferral: the requests arrived but not dispatched, then the batch, in index
// order, split three ways (stable): a bound available by s (the arrival plus
// the prediction delay) -> the dispatch policy; waited beta steps past
// arrival without one, or the last dispatch step -> round robin; otherwise
// they keep waiting for the next dispatch step.
__global__ void __launch_bounds__(kSt, 1)
stream_select_kernel(int64_t lo, int nb, int64_t hi, int32_t beta, int last, const int64_t *arrival,
                     const int32_t *pred_delay, const int32_t *pend_in, int32_t *pend_out,
                     int32_t *cid, int32_t *tout, StreamState *S) {
  pdl_prologue();
  __shared__ int s_w[kStWarps];
  const long long s = arrival[hi - 1];
  const int np = S->npend, n = np + nb;
  int nc = 0, nt = 0, nk = 0;
  for (int c0 = 0; c0 < n; c0 += kSt) {
    const int x = c0 + static_cast<int>(threadIdx.x);
    int id = -1;
    bool av = false, to = false, kp = false;
    if (x < n) {
      id = x < np ? pend_in[x] : static_cast<int>(lo + (x - np));
      av = arrival[id] + pred_delay[id] <= s;
      to = !av && (arrival[id] + beta <= s || last);
      kp = !av && !to;
    }
    int tc, tt, tk;
    const int pc = block_flag_scan(av, s_w, tc);
    const int pt = block_flag_scan(to, s_w, tt);
    const int pk = block_flag_scan(kp, s_w, tk);
    if (av) cid[nc + pc] = id;
    if (to) tout[nt + pt] = id;
    if (kp) pend_out[nk + pk] = id;
    nc += tc;
    nt += tt;
    nk += tk;
  }
  if (threadIdx.x == 0) {
    S->nc = nc;
    S->nto = nt;
    S->npend = nk;
  }
}

// 2. Completions, sorted by (step, id), enter the ring of the last Wn; the
//    c-th completion ever goes to slot c mod Wn.
__global__ void stream_window_kernel(int ndone, long long c0, int Wn, const int32_t *perm,
                                     const int32_t *done_id, const int32_t *true_len,
                                     const int32_t *pred, int32_t *win_true, int32_t *win_pred) {
  pdl_prologue();
  const int stride = gridDim.x * blockDim.x;
  for (int x = blockIdx.x * blockDim.x + threadIdx.x; x < ndone; x += stride) {
    if (x < ndone - Wn) continue;  // overwritten by a later completion of this batch
    const int id = done_id[perm[x]];
    const int slot = static_cast<int>((c0 + x) % Wn);
    win_true[slot] = true_len[id];
    win_pred[slot] = pred[id];
  }
}

// 3. Predictions of the requests in the system, then of the candidates
//    (the batch lo.., or the listed ids, whose prompts are gathered too).
__global__ void stream_gather_kernel(int nact, int nb, int64_t lo, const int32_t *act,
                                     const int32_t *cid, const int32_t *pred,
                                     const int32_t *prompt, int32_t *qpred, int32_t *cp) {
  pdl_prologue();
  const int stride = gridDim.x * blockDim.x;
  for (int x = blockIdx.x * blockDim.x + threadIdx.x; x < nact + nb; x += stride) {
    if (x < nact) {
      qpred[x] = pred[act[x]];
    } else {
      const int id = cid ? cid[x - nact] : static_cast<int>(lo + (x - nact));
      qpred[x] = pred[id];
      if (cid) cp[x - nact] = prompt[id];
    }
  }
}

// 3'. No bound available: U = prediction, the batch goes round robin.  With
//     set_u = 0 only the choices (the round-robin dispatch policy).
//     choice[x] is candidate x's: lo + x, or the listed cid[x].
__global__ void stream_rr_kernel(int n, int nb, int64_t lo, int D, int set_u, const int32_t *qpred,
                                 int32_t *Uq, const int32_t *cid, int32_t *choice) {
  pdl_prologue();
  const int stride = gridDim.x * blockDim.x;
  for (int x = blockIdx.x * blockDim.x + threadIdx.x; x < n; x += stride) {
    if (set_u) Uq[x] = qpred[x];
    if (x < nb) choice[x] = static_cast<int32_t>((cid ? static_cast<int64_t>(cid[x]) : lo + x) % D);
  }
}

// 5'. Least requests (one warp): candidate j goes to the decoder with the
//     fewest requests in the system, counting the batch's earlier choices;
//     ties to the lowest index.  Lane l keeps the counts of decoders l, l + 32,
//     ... in shared memory; per candidate two warp minima give the smallest
//     count and then the lowest decoder holding it.
__global__ void stream_lr_kernel(int D, int nb, const int64_t *res_off, int32_t *choice) {
  pdl_prologue();
  __shared__ uint32_t s_c[kStreamMaxD];
  const int lane = threadIdx.x;
  for (int k = lane; k < D; k += 32) s_c[k] = static_cast<uint32_t>(res_off[k + 1] - res_off[k]);
  __syncwarp();
  for (int j = 0; j < nb; ++j) {
    uint32_t c = 0xffffffffu, ck = 0xffffffffu;  // this lane's smallest count, its lowest decoder
    for (int k = lane; k < D; k += 32)
      if (s_c[k] < c) {
        c = s_c[k];
        ck = static_cast<uint32_t>(k);
      }
    const uint32_t cmin = __reduce_min_sync(0xffffffffu, c);
    const uint32_t bk = __reduce_min_sync(0xffffffffu, c == cmin ? ck : 0xffffffffu);
    if (lane == 0) {
      choice[j] = static_cast<int32_t>(bk);
      s_c[bk] = cmin + 1;
    }
    __syncwarp();
  }
}

// 4. Residents by decoder (running with g, waiting with g = 0) and the
//    waiting count per decoder; new bounds of the requests in the system.
__global__ void __launch_bounds__(kSt, 1)
//    Under deferral a request whose prediction is not in by s (arrival +
//    delay > s) is bounded by the horizon H.
stream_csr_kernel(int nact, int D, int rr, const int32_t *q_dev, int32_t *q_out_b,
                  const int32_t *act, const uint8_t *st, const int32_t *g, const int32_t *dec,
                  const int32_t *prompt, int32_t *Uq, int32_t *U, int64_t *res_off,
                  int32_t *rp, int32_t *rg, int32_t *rU, int32_t *Q, const int64_t *arrival,
                  const int32_t *pred_delay, int64_t hi, int32_t H) {
  pdl_prologue();
  if (pred_delay != nullptr) {  // before anything reads Uq
    const long long s = arrival[hi - 1];
    for (int x = threadIdx.x; x < nact; x += kSt) {
      const int id = act[x];
      if (arrival[id] + pred_delay[id] > s) Uq[x] = H;
    }
    __syncthreads();
  }
  __shared__ int s_cnt[kStreamMaxD], s_q[kStreamMaxD], s_cur[kStreamMaxD];
  __shared__ int s_w[kStWarps];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int k = tid; k < D; k += kSt) s_cnt[k] = s_q[k] = 0;
  __syncthreads();
  for (int x = tid; x < nact; x += kSt) {
    const int id = act[x];
    U[id] = Uq[x];
    atomicAdd(&s_cnt[dec[id]], 1);
    if (st[id] == kWaiting) atomicAdd(&s_q[dec[id]], 1);
  }
  __syncthreads();
  const int c = tid < D ? s_cnt[tid] : 0;  // D <= kSt
  int incl = c;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += y;
  }
  if (lane == 31) s_w[warp] = incl;
  __syncthreads();
  int base = 0;
  for (int w = 0; w < warp; ++w) base += s_w[w];
  if (tid < D) {
    const int ex = base + incl - c;
    s_cur[tid] = ex;
    res_off[tid] = ex;
    Q[tid] = s_q[tid];
    if (tid == D - 1) res_off[D] = ex + c;
  }
  __syncthreads();
  for (int x = tid; x < nact; x += kSt) {
    const int id = act[x];
    const int pos = atomicAdd(&s_cur[dec[id]], 1);
    rp[pos] = prompt[id];
    rg[pos] = st[id] == kRunning ? g[id] : 0;
    rU[pos] = Uq[x];
  }
  if (tid == 0) *q_out_b = rr ? -1 : q_dev[0];
}

// 5. (shared-memory form) SEQUENTIAL dispatch of the batch without a dense K.
// Decoder k's occupancy is held as its residents' pairs (e, b), sorted by e:
// on a step t the live residents are those with e > t, so
//   K_k(t) + t = S(t) + t (C(t) + 1),  S / C = b-sum / count of e > t,
// which is linear and rising between consecutive end steps.  Its maximum over
// t < u is therefore taken at t = e_i - 1 for some e_i <= u, or at t = u - 1:
// with the pairs sorted ascending and S_i / C_i the sums over pairs i.. n-1,
//   M_k(u) = max( max_{e_i <= u} S_i + (e_i - 1)(C_i + 1),
//                 S' + (u - 1)(C' + 1) ),  S' / C' over the pairs with e > u.
// (A pair tied on e with one before it gives a value no larger than the
// first's, so ties need no merging.)  Beside the sorted pairs each decoder
// keeps the suffix sums of b and the prefix maxima of the first term, so a
// score is a binary search for the pairs with e <= u and two reads.  One warp
// walks the batch: a lane scores a decoder, the warp picks (feasible with the
// smallest Q, else the largest headroom, ties to the lowest index), inserts
// (u, p + 1) into the chosen decoder's list and rebuilds its tables.  The
// decisions and range errors are those of the dense projection followed by
// maps_dispatch SEQUENTIAL.
// Shared memory: the pool of pairs (the residents of decoder k plus room for
// nb reservations at base_k = res_off[k] + k nb), the unsorted pairs, and the
// per-decoder tables.
// The packed decision key, the smallest wins: a feasible decoder (h >= 0)
// ranks by Q, an infeasible one after every feasible one by the deficit -h,
// each then by index: inf << 63 | v << 10 | k.  mc (the max-headroom rule)
// ranks every decoder as the infeasible class does, by -h: v = 2^33 - h is
// positive (h <= cap < 2^31) and, like the deficit, below 2^53 for any M the
// walk forms.
__device__ __forceinline__ unsigned long long dispatch_key(long long h, int q, int k, int mc) {
  const bool feas = h >= 0 && !mc;
  const unsigned long long v = feas ? static_cast<unsigned long long>(q)
                               : mc ? static_cast<unsigned long long>((1ll << 33) - h)
                                    : static_cast<unsigned long long>(-h);
  return (feas ? 0ull : 1ull << 63) | (v << 10) | static_cast<unsigned>(k);
}

size_t stream_dispatch_smem(int D, int nact, int nb) {
  const size_t pool = static_cast<size_t>(nact) + static_cast<size_t>(D) * nb;
  return 16 * pool + 8 * static_cast<size_t>(nact) + 16 * static_cast<size_t>(D) +
         12 * static_cast<size_t>(nb) + 64;
}

// A decoder's tables from its sorted pairs (one warp): SS[i] = sum of b over
// pairs i.. n-1, and PM[i] = the largest V over pairs 0..i, with
// V_i = SS[i] + (E[i] - 1)(n - i + 1) (K + t at t = E[i] - 1).  Returns
// whether some K(t) exceeds INT32_MAX (the projection's range error); below
// that every SS, V and PM fits 32 bits.
// Barrier `id` over the first `count` threads (whole warps) of the block.
__device__ __forceinline__ void named_bar(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ bool rebuild_tables(const int32_t *E, const int32_t *Bv, uint32_t *SS, uint32_t *PM,
                               int n) {
  const int lane = threadIdx.x & 31;
  unsigned long long carry = 0;
  bool over = false;
  for (int r = (n - 1) >> 5; r >= 0; --r) {  // suffix sums, last round first
    const int i = r * 32 + lane;
    const unsigned long long b = i < n ? static_cast<unsigned long long>(Bv[i]) : 0ull;
    unsigned long long suf = b;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const unsigned long long y = __shfl_down_sync(0xffffffffu, suf, off);
      if (lane + off < 32) suf += y;
    }
    if (i < n) {
      const unsigned long long ss = suf + carry;
      // K at the segment's last step: the pairs i.. n-1 are live there
      over |= ss + static_cast<unsigned long long>(E[i] - 1) * (n - i) > 0x7fffffffull;
      SS[i] = static_cast<uint32_t>(ss);
    }
    carry += __shfl_sync(0xffffffffu, suf, 0);
  }
  __syncwarp();
  uint32_t run = 0;
  for (int r = 0; r <= (n - 1) >> 5; ++r) {  // prefix maxima, first round first
    const int i = r * 32 + lane;
    uint32_t incl = i < n ? SS[i] + static_cast<uint32_t>(E[i] - 1) * static_cast<uint32_t>(n - i + 1) : 0u;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl = max(incl, y);
    }
    incl = max(incl, run);
    if (i < n) PM[i] = incl;
    run = __shfl_sync(0xffffffffu, incl, 31);
  }
  __syncwarp();
  return __any_sync(0xffffffffu, over);
}

__global__ void __launch_bounds__(kSt, 1)
stream_dispatch_kernel(int D, int H, int nb, int mc, const int64_t *res_off, const int32_t *rp,
                       const int32_t *rg, const int32_t *rU, const int32_t *capv, int32_t *Q,
                       const int32_t *cp, const int32_t *cU, int32_t *choice, int64_t *headroom,
                       int32_t *status) {
  pdl_prologue();
  extern __shared__ __align__(16) unsigned char sdm[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nact = static_cast<int>(res_off[D]);
  const int pool = nact + D * nb;
  int32_t *E = reinterpret_cast<int32_t *>(sdm);           // [pool] sorted end steps
  int32_t *Bv = E + pool;                                  // [pool] their b
  uint32_t *SS = reinterpret_cast<uint32_t *>(Bv + pool);  // [pool] suffix sums of b
  uint32_t *PM = SS + pool;                                // [pool] prefix maxima of V
  int32_t *uE = reinterpret_cast<int32_t *>(PM + pool);    // [nact] unsorted
  int32_t *uB = uE + nact;
  int32_t *s_base = uB + nact, *s_n = s_base + D, *s_q = s_n + D, *s_cap = s_q + D;
  int32_t *s_cp = s_cap + D, *s_cu = s_cp + nb;            // [nb] the batch
  int32_t *s_ch = s_cu + nb;                               // [nb] choices (fast path)
  __shared__ int s_bad, s_fast;
  if (tid == 0) {
    s_bad = 0;
    s_fast = 0;
  }
  __syncthreads();
  for (int k = tid; k < D; k += kSt) {
    const int lo = static_cast<int>(res_off[k]);
    s_base[k] = lo + k * nb;
    s_n[k] = static_cast<int>(res_off[k + 1]) - lo;
    s_q[k] = Q[k];
    s_cap[k] = capv[k];
    if ((s_q[k] | s_cap[k]) < 0) s_bad = 1;
  }
  for (int j = tid; j < nb; j += kSt) {
    s_cp[j] = cp[j];
    s_cu[j] = cU[j];
  }
  for (int x = tid; x < nact; x += kSt) {  // the residents' pairs, as the projection forms them
    const int32_t p = rp[x], g = rg[x], U = rU[x];
    int32_t e = 1, b = 0;
    if ((p | g | U) < 0) {
      s_bad = 1;
    } else {
      const long long bb = static_cast<long long>(p) + g + 1;
      if (bb > 0x7fffffffLL) s_bad = 1;
      b = static_cast<int32_t>(bb > 0x7fffffffLL ? 0x7fffffffLL : bb);
      e = U - g;
      e = e < 1 ? 1 : (e > H ? H : e);
    }
    uE[x] = e;
    uB[x] = b;
  }
  __syncthreads();
  // Without a headroom output and with the Q-first rule, a decoder whose peak
  // is provably within its capacity is decided by (Q, index) alone.
  const bool quick = headroom == nullptr && mc == 0;
  // Fast path (at most 32 decoders, no headroom output, Q-first rule): the
  // choices by (Q, index) alone, taken when every decoder is shown feasible at
  // every step, before any list is sorted.  For t < u,
  // K(t) + t = S(t) + t (C(t) + 1) with S <= the decoder's b-sum and C <= n
  // while t < e_max, and K(t) + t = t after e_max, so decoder k's peak for a
  // candidate of horizon u, after the batch's earlier reservations on k, is
  // at most
  //   max(b-sum + (min(u, e_max) - 1)(n + 1), u - 1)
  //   + the sum of p + u over those reservations
  // (each adds p + t + 1 for t < u).  While p + 1 + that bound <= cap for
  // every decoder, every decoder is feasible, so the rule picks the smallest
  // (Q, index), which is the choice taken: the decisions are the walk's, and
  // the lists need no sorting.  If some decoder might not fit at some step
  // the walk decides the whole batch (Q is written only on success).
  // The picks of the Q-first rule have a closed form: taking the smallest
  // (Q, index) and raising that Q by one, level by level, at level L every
  // decoder with Q <= L takes one candidate, in index order.  So candidate j
  // goes to level L, the smallest with cum(L) > j where
  // cum(L) = sum over k of max(0, L - Q_k + 1), and there to the
  // (j - cum(L - 1))-th decoder with Q <= L.  Each candidate's pick is found
  // on its own; then one warp per decoder sums the reservations before each
  // candidate (a scan) and checks the bound.
  if (quick && D <= 32) {
    __shared__ long long f_sb[32];
    __shared__ int f_em[32], f_cnt[32], f_inv, f_miss;
    if (tid == 0) {
      f_inv = 0;
      f_miss = 0;
    }
    __syncthreads();
    if (warp < D) {  // decoder `warp`: its residents' b-sum and largest end step
      const int k = warp, n = s_n[k], lo = s_base[k] - k * nb;
      long long sb = 0;
      int em = 1;
      for (int i = lane; i < n; i += 32) {
        sb += uB[lo + i];
        em = max(em, uE[lo + i]);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        sb += __shfl_xor_sync(0xffffffffu, sb, off);
        em = max(em, __shfl_xor_sync(0xffffffffu, em, off));
      }
      if (lane == 0) {
        f_sb[k] = sb;
        f_em[k] = em;
        f_cnt[k] = 0;
        // checked once: every Q stays within 21 bits (a Q grows by at most
        // nb), and no K of the residents reaches INT32_MAX (so the tables'
        // range checks could not fire); otherwise the walk handles the batch
        if (static_cast<long long>(s_q[k]) + nb >= (1 << 21) ||
            sb + static_cast<long long>(em - 1) * (n + 1) > 0x7fffffffLL)
          f_inv = 1;
      }
    }
    for (int j = tid; j < nb; j += kSt)
      if ((s_cp[j] | s_cu[j]) < 0) f_inv = 1;  // every candidate valid
    __syncthreads();
    if (!f_inv) {
      int qmin = 0x7fffffff;
      for (int k = 0; k < D; ++k) qmin = min(qmin, s_q[k]);
      auto cum = [&](int L) {  // picks made by the end of level L
        int c = 0;
        for (int k = 0; k < D; ++k) c += max(0, L - s_q[k] + 1);
        return c;
      };
      for (int j = tid; j < nb; j += kSt) {
        // the decoder at qmin alone takes nb picks by level qmin + nb - 1
        int lo = qmin, hi = qmin + nb - 1;
        while (lo < hi) {
          const int mid = lo + (hi - lo) / 2;
          if (cum(mid) > j)
            hi = mid;
          else
            lo = mid + 1;
        }
        int r = j - (lo > qmin ? cum(lo - 1) : 0);
        int pick = -1;
        for (int k = 0; k < D; ++k)
          if (s_q[k] <= lo && r-- == 0) {
            pick = k;
            break;
          }
        s_ch[j] = pick < 0 ? 0 : pick;
        if (pick < 0) f_miss = 1;  // cannot happen; the walk would decide the batch
      }
    }
    __syncthreads();
    if (!f_inv && warp < D) {
      const int k = warp, n = s_n[k], em = f_em[k];
      const long long sb = f_sb[k], cap = s_cap[k];
      long long carry = 0;  // p + u of this decoder's reservations so far
      int cnt = 0;
      bool miss = false;
      for (int j0 = 0; j0 < nb; j0 += 32) {
        const int j = j0 + lane;
        const bool ok = j < nb;
        const int32_t p = ok ? s_cp[j] : 0, U = ok ? s_cu[j] : 1;
        const int u = U < 1 ? 1 : (U > H ? H : U);
        const bool mine = ok && s_ch[j] == k;
        const long long w = mine ? static_cast<long long>(p) + u : 0;
        long long incl = w;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const long long y = __shfl_up_sync(0xffffffffu, incl, off);
          if (lane >= off) incl += y;
        }
        const long long add = carry + incl - w;  // the reservations before candidate j
        const long long b0 = max(sb + static_cast<long long>(min(u, em) - 1) * (n + 1),
                                 static_cast<long long>(u - 1));
        miss |= ok && static_cast<long long>(p) + 1 + b0 + add > cap;
        carry += __shfl_sync(0xffffffffu, incl, 31);
        cnt += __popc(__ballot_sync(0xffffffffu, mine));
      }
      if (__any_sync(0xffffffffu, miss) && lane == 0) f_miss = 1;
      if (lane == 0) f_cnt[k] = cnt;
    }
    __syncthreads();
    const bool fits = !f_inv && !f_miss;
    if (fits) {
      for (int j = tid; j < nb; j += kSt) choice[j] = s_ch[j];
      for (int k = tid; k < D; k += kSt) s_q[k] += f_cnt[k];
    }
    if (tid == 0) s_fast = fits ? 1 : 0;
  }
  __syncthreads();

  if (!s_fast) {
    // sort each decoder's pairs by e (rank among the decoder's pairs, ties by
    // position), and check sum b <= INT32_MAX (K at step 0)
    for (int k = warp; k < D; k += kSt / 32) {
      const int lo = s_base[k] - k * nb, n = s_n[k], base = s_base[k];
      long long sb = 0;
      for (int i = lane; i < n; i += 32) {
        const int ei = uE[lo + i];
        int r = 0;
        for (int j2 = 0; j2 < n; ++j2) {
          const int ej = uE[lo + j2];
          r += ej < ei || (ej == ei && j2 < i);
        }
        E[base + r] = ei;
        Bv[base + r] = uB[lo + i];
        sb += uB[lo + i];
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sb += __shfl_xor_sync(0xffffffffu, sb, off);
      if (lane == 0 && sb > 0x7fffffffLL) s_bad = 1;
      __syncwarp();  // the sorted pairs are written
      if (rebuild_tables(E + base, Bv + base, SS + base, PM + base, n) && lane == 0) s_bad = 1;
    }
    __syncthreads();
  }
  if (tid == 0 && s_bad) flag_error(status, MAPS_E_RANGE);

  // The walk: one warp, no block barrier.  Lane l scores decoders l, l + 32,
  // ...: a binary search over the decoder's sorted ends gives c (the pairs with
  // e <= u), then M = max(PM[c - 1], SS[c] + (u - 1)(n - c + 1)); a packed key
  // picks (feasible first, then Q or the largest headroom, then the lowest
  // index); the warp inserts the footprint and rebuilds that decoder's tables.
  if (s_fast) {
    // decided by the fast path
  } else if (D <= 32) {
    // Two warps, one decoder per lane.  Warp 0 holds each decoder's list
    // length, base, Q and capacity in registers, scores the candidates, picks
    // and books each decision and hands it to warp 1 through shared memory
    // (named barrier 1); warp 1 inserts the reservation into the chosen
    // decoder's list and scores that decoder again for the next candidate
    // (named barrier 2).  Meanwhile warp 0 scores the next candidate on the
    // lists as they stand: a reservation only raises the chosen decoder's Q
    // and occupancy, so every other decoder's key is already final and the
    // chosen one's is replaced by warp 1's.  Keys: inf << 63 | v << 10 | k,
    // the smallest wins.
    __shared__ int h_bk, h_pos, h_n, h_base, h_q, h_cap, h_c;
    __shared__ long long h_M;
    __shared__ unsigned long long h_key;
    auto clampu = [&](int32_t U) { return U < 1 ? 1 : (U > H ? H : U); };
    // c = the pairs with e <= u of a sorted list (8-ary search: eight
    // independent probes per level, one level for up to 8 pairs)
    auto count_le = [&](const int32_t *Ek, int n, int u) {
      int lo = 0, hi = n;
      while (lo < hi) {
        const int len = hi - lo;
        int nlo = lo, nhi = hi;
#pragma unroll
        for (int i = 0; i < 8; ++i) {  // probes cover every position when len <= 8
          const int pi = lo + (len * i) / 8;
          if (Ek[pi] <= u)
            nlo = max(nlo, pi + 1);
          else
            nhi = min(nhi, pi);
        }
        lo = nlo;
        hi = nhi;
      }
      return lo;
    };
    auto key_of = [mc](int k, int q, int cap, int32_t p, long long M) {
      const long long h = static_cast<long long>(cap) - (static_cast<long long>(p) + 1 + M);
      return dispatch_key(h, q, k, mc);
    };
    if (warp == 0) {
      const int k = lane;
      const bool has = k < D;
      int n_r = has ? s_n[k] : 0, q_r = has ? s_q[k] : 0;
      const int base_r = has ? s_base[k] : 0, cap_r = has ? s_cap[k] : 0;
      bool bad = false, have = false;  // have: key, c and M are the current candidate's
      unsigned long long key = ~0ull;
      long long M = 0;
      int c = 0;
      auto score = [&](int32_t pp, int uu) {
        key = ~0ull;
        if (!has) return;
        if (quick && n_r > 0) {
          const long long mub = max(static_cast<long long>(PM[base_r + n_r - 1]),
                                    static_cast<long long>(SS[base_r]) +
                                        static_cast<long long>(uu - 1) * (n_r + 1));
          if (static_cast<long long>(pp) + 1 + mub <= cap_r) {
            key = (static_cast<unsigned long long>(q_r) << 10) | static_cast<unsigned>(k);
            c = -1;   // found at insertion
            M = mub;  // bounds every new cell: no range error (cap <= INT32_MAX)
            return;
          }
        }
        c = count_le(E + base_r, n_r, uu);
        const long long full = c > 0 ? static_cast<long long>(PM[base_r + c - 1]) : LLONG_MIN;
        const long long part = static_cast<long long>(c < n_r ? SS[base_r + c] : 0u) +
                               static_cast<long long>(uu - 1) * (n_r - c + 1);
        M = max(full, part);
        key = key_of(k, q_r, cap_r, pp, M);
      };
      for (int j = 0; j < nb; ++j) {
        const int32_t p = s_cp[j], U = s_cu[j];
        int bk = -1;
        if ((p | U) >= 0) {
          if (!have) score(p, clampu(U));
          // the warp's smallest key: one 32-bit reduction when every value
          // fits 21 bits (inf << 31 | v << 10 | k, the same order), else a ladder
          const unsigned long long kv = (key >> 10) & ((1ull << 53) - 1);
          const bool none = key == ~0ull;
          if (__all_sync(0xffffffffu, none || kv < (1ull << 21))) {
            const uint32_t k32 = none ? 0xffffffffu
                                      : (static_cast<uint32_t>(key >> 63) << 31) |
                                            (static_cast<uint32_t>(kv) << 10) | static_cast<uint32_t>(key & 1023u);
            bk = static_cast<int>(__reduce_min_sync(0xffffffffu, k32) & 1023u);
          } else {
            unsigned long long kk = key;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
              const unsigned long long o = __shfl_xor_sync(0xffffffffu, kk, off);
              kk = o < kk ? o : kk;
            }
            bk = static_cast<int>(kk & 1023u);
          }
          if (lane == bk) {  // the chosen decoder's lane books the decision
            choice[j] = bk;
            if (headroom) headroom[j] = static_cast<long long>(cap_r) - (static_cast<long long>(p) + 1 + M);
            bad |= q_r == 0x7fffffff;
            q_r += q_r == 0x7fffffff ? 0 : 1;
            // every new cell K + p + t + 1 (t < u) is at most M + p + 1
            bad |= static_cast<long long>(p) + 1 + M > 0x7fffffffLL;
            h_bk = bk;
            h_pos = c;
            h_n = n_r;
            h_base = base_r;
            h_q = q_r;
            h_cap = cap_r;
            n_r += 1;
          }
        } else if (lane == 0) {
          bad = true;
          choice[j] = -1;
          if (headroom) headroom[j] = 0;
          h_bk = -1;
        }
        named_bar(1, 64);  // the decision goes to warp 1
        const bool nxt = j + 1 < nb;
        const int32_t p1 = nxt ? s_cp[j + 1] : 0, U1 = nxt ? s_cu[j + 1] : 0;
        const bool ok1 = nxt && (p1 | U1) >= 0;
        if (ok1) score(p1, clampu(U1));  // the chosen decoder's key is replaced below
        named_bar(2, 64);  // warp 1 has updated the list and scored it again
        if (ok1 && lane == bk) {
          key = h_key;
          c = h_c;
          M = h_M;
        }
        have = ok1;
      }
      if (__any_sync(0xffffffffu, bad) && lane == 0) flag_error(status, MAPS_E_RANGE);
      if (has) {
        s_n[k] = n_r;
        s_q[k] = q_r;
      }
    } else if (warp == 1) {
      for (int j = 0; j < nb; ++j) {
        named_bar(1, 64);
        const int bk = h_bk;
        if (bk >= 0) {
          const int n = h_n, base = h_base, m = n + 1;
          const int32_t p = s_cp[j];
          const int u = clampu(s_cu[j]);
          int pos = h_pos;  // -1: the scoring took the bound, count the pairs with e <= u here
          if (pos < 0) {
            if (n < 32)
              pos = __popc(__ballot_sync(0xffffffffu, lane < n && E[base + lane] <= u));
            else
              pos = count_le(E + base, n, u);
          }
          const bool nxt = j + 1 < nb;
          const int32_t p1 = nxt ? s_cp[j + 1] : 0, U1 = nxt ? s_cu[j + 1] : 0;
          const bool ok1 = nxt && (p1 | U1) >= 0;
          const int u1 = clampu(U1);
          int c1 = 0;
          long long M1 = 0;
          if (m <= 32) {
            // one round: lane i takes pair i of the new list; the suffix sums
            // follow from the old ones (b more before the new pair, the same
            // after it) and one shuffle scan gives the prefix maxima of V, in
            // 32 bits (the booking's check keeps every K + t within INT32_MAX)
            const int src = lane <= pos ? lane : lane - 1;
            const bool old_ok = src < n;
            const int eo = old_ok ? E[base + src] : 0, bo = old_ok ? Bv[base + src] : 0;
            const uint32_t so = old_ok ? SS[base + src] : 0u;
            const uint32_t bnew = static_cast<uint32_t>(p) + 1u;
            const int e2 = lane == pos ? u : eo;
            const int b2 = lane == pos ? static_cast<int>(bnew) : bo;
            const uint32_t suf = lane <= pos ? so + bnew : so;
            uint32_t V = lane < m ? suf + static_cast<uint32_t>(e2 - 1) * static_cast<uint32_t>(m - lane + 1) : 0u;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
              const uint32_t y = __shfl_up_sync(0xffffffffu, V, off);
              if (lane >= off) V = max(V, y);
            }
            __syncwarp();  // every lane has read the old list
            if (lane < m) {
              E[base + lane] = e2;
              Bv[base + lane] = b2;
              SS[base + lane] = suf;
              PM[base + lane] = V;
            }
            // the new list's count and table values at the next candidate's u
            c1 = __popc(__ballot_sync(0xffffffffu, lane < m && e2 <= u1));
            const uint32_t pmb = __shfl_sync(0xffffffffu, V, c1 > 0 ? c1 - 1 : 0);
            const uint32_t ssb = __shfl_sync(0xffffffffu, suf, c1 < m ? c1 : 0);
            const long long full = c1 > 0 ? static_cast<long long>(pmb) : LLONG_MIN;
            const long long part = static_cast<long long>(c1 < m ? ssb : 0u) +
                                   static_cast<long long>(u1 - 1) * (m - c1 + 1);
            M1 = max(full, part);
          } else {
            // a list past 32 pairs: shift [pos, n) up by one (last round
            // first), place the new pair, rebuild the tables
            for (int r = (n - 1) >> 5; r >= 0; --r) {
              const int i = r * 32 + lane;
              const bool mv = i < n && i >= pos;
              const int e = mv ? E[base + i] : 0, b = mv ? Bv[base + i] : 0;
              __syncwarp();
              if (mv) {
                E[base + i + 1] = e;
                Bv[base + i + 1] = b;
              }
              __syncwarp();
            }
            if (lane == 0) {
              E[base + pos] = u;
              Bv[base + pos] = p + 1;
            }
            __syncwarp();
            rebuild_tables(E + base, Bv + base, SS + base, PM + base, m);
            if (ok1) {
              c1 = count_le(E + base, m, u1);
              const long long full = c1 > 0 ? static_cast<long long>(PM[base + c1 - 1]) : LLONG_MIN;
              const long long part = static_cast<long long>(c1 < m ? SS[base + c1] : 0u) +
                                     static_cast<long long>(u1 - 1) * (m - c1 + 1);
              M1 = max(full, part);
            }
          }
          if (ok1 && lane == 0) {
            h_key = key_of(bk, h_q, h_cap, p1, M1);
            h_c = c1;
            h_M = M1;
          }
        }
        named_bar(2, 64);
      }
    }
  } else if (warp == 0) {
    for (int j = 0; j < nb; ++j) {
      const int32_t p = s_cp[j], U = s_cu[j];
      if ((p | U) < 0) {
        if (lane == 0) {
          flag_error(status, MAPS_E_RANGE);
          choice[j] = -1;
          if (headroom) headroom[j] = 0;
        }
        continue;
      }
      const int u = U < 1 ? 1 : (U > H ? H : U);
      unsigned long long key = ~0ull;  // inf << 63 | v << 10 | k, the smallest wins
      long long bM = 0;                // M and c of this lane's best decoder
      int bc = 0;
      for (int k = lane; k < D; k += 32) {
        const int n = s_n[k], base = s_base[k];
        if (quick && n > 0) {  // a sure fit is decided by (Q, index) alone
          const long long mub = max(static_cast<long long>(PM[base + n - 1]),
                                    static_cast<long long>(SS[base]) +
                                        static_cast<long long>(u - 1) * (n + 1));
          if (static_cast<long long>(p) + 1 + mub <= s_cap[k]) {
            const unsigned long long kk = (static_cast<unsigned long long>(s_q[k]) << 10) |
                                          static_cast<unsigned>(k);
            if (kk < key) {
              key = kk;
              bM = mub;
              bc = -1;
            }
            continue;
          }
        }
        int lo = 0, hi = n;  // c = the pairs with e <= u
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (E[base + mid] <= u)
            lo = mid + 1;
          else
            hi = mid;
        }
        const int c = lo;
        const long long full = c > 0 ? static_cast<long long>(PM[base + c - 1]) : LLONG_MIN;
        const long long part = static_cast<long long>(c < n ? SS[base + c] : 0u) +
                               static_cast<long long>(u - 1) * (n - c + 1);
        const long long M = max(full, part);
        const long long h = static_cast<long long>(s_cap[k]) - (static_cast<long long>(p) + 1 + M);
        const unsigned long long kk = dispatch_key(h, s_q[k], k, mc);
        if (kk < key) {
          key = kk;
          bM = M;
          bc = c;
        }
      }
      // The warp's smallest key.  When every value fits 21 bits the key packs
      // into 32 (inf << 31 | v << 10 | k, the same order) and one reduction
      // finds it; otherwise a shuffle ladder over the 64-bit keys.
      const unsigned long long kv = (key >> 10) & ((1ull << 53) - 1);
      const bool none = key == ~0ull;  // a lane without decoders
      int bk;
      if (__all_sync(0xffffffffu, none || kv < (1ull << 21))) {
        const uint32_t k32 = none ? 0xffffffffu
                                  : (static_cast<uint32_t>(key >> 63) << 31) |
                                        (static_cast<uint32_t>(kv) << 10) | static_cast<uint32_t>(key & 1023u);
        bk = static_cast<int>(__reduce_min_sync(0xffffffffu, k32) & 1023u);
      } else {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const unsigned long long o = __shfl_xor_sync(0xffffffffu, key, off);
          key = o < key ? o : key;
        }
        bk = static_cast<int>(key & 1023u);
      }
      // the winner's lane (decoder bk is lane bk % 32's) hands over M and c
      const long long Mb = __shfl_sync(0xffffffffu, bM, bk & 31);
      int pos = __shfl_sync(0xffffffffu, bc, bk & 31);
      const int n = s_n[bk], base = s_base[bk];
      if (pos < 0) {  // the bound decided it: the pairs with e <= u place the new one
        int lo = 0, hi = n;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (E[base + mid] <= u)
            lo = mid + 1;
          else
            hi = mid;
        }
        pos = lo;
      }
      if (lane == 0) {
        choice[j] = bk;
        if (headroom) headroom[j] = static_cast<long long>(s_cap[bk]) - (static_cast<long long>(p) + 1 + Mb);
        if (s_q[bk] == 0x7fffffff)
          flag_error(status, MAPS_E_RANGE);
        else
          s_q[bk] += 1;
        // every new cell K + p + t + 1 (t < u) is at most M + p + 1
        if (static_cast<long long>(p) + 1 + Mb > 0x7fffffffLL) flag_error(status, MAPS_E_RANGE);
      }
      // reserve: (u, p + 1) joins decoder bk's pairs after those with e <= u
      const int m = n + 1;
      if (m <= 32) {
        // One round: lane i takes pair i of the new list.  The suffix sums
        // follow from the old ones (b more before the new pair, the same
        // after it), and the prefix maxima of V take one shuffle scan, in 32
        // bits (the check above keeps every K + t of the new list within
        // INT32_MAX).
        const int src = lane <= pos ? lane : lane - 1;  // the old pair this lane keeps
        const bool old_ok = src < n;
        const int eo = old_ok ? E[base + src] : 0, bo = old_ok ? Bv[base + src] : 0;
        const uint32_t so = old_ok ? SS[base + src] : 0u;
        const uint32_t bnew = static_cast<uint32_t>(p) + 1u;
        const int e2 = lane == pos ? u : eo;
        const int b2 = lane == pos ? static_cast<int>(bnew) : bo;
        const uint32_t suf = lane <= pos ? so + bnew : so;
        uint32_t V = lane < m ? suf + static_cast<uint32_t>(e2 - 1) * static_cast<uint32_t>(m - lane + 1) : 0u;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, V, off);
          if (lane >= off) V = max(V, y);
        }
        __syncwarp();  // every lane has read the old list
        if (lane < m) {
          E[base + lane] = e2;
          Bv[base + lane] = b2;
          SS[base + lane] = suf;
          PM[base + lane] = V;
        }
        if (lane == 0) s_n[bk] = m;
        __syncwarp();
        continue;
      }
      for (int r = (n - 1) >> 5; r >= 0; --r) {  // shift [pos, n) up by one, last round first
        const int i = r * 32 + lane;
        const bool mv = i < n && i >= pos;
        const int e = mv ? E[base + i] : 0, b = mv ? Bv[base + i] : 0;
        __syncwarp();
        if (mv) {
          E[base + i + 1] = e;
          Bv[base + i + 1] = b;
        }
        __syncwarp();
      }
      if (lane == 0) {
        E[base + pos] = u;
        Bv[base + pos] = p + 1;
        s_n[bk] = n + 1;
      }
      __syncwarp();
      rebuild_tables(E + base, Bv + base, SS + base, PM + base, n + 1);
    }
  }
  __syncthreads();
  for (int k = tid; k < D; k += kSt) Q[k] = s_q[k];
}

// 5''. Deferral: the listed requests join the waiting queues at act[nact..]:
//      with choices cch (and bounds Uq[nact + i]), or, with cch null, round
//      robin with the horizon as their bound (timed out without one).
__global__ void stream_enqueue_list_kernel(int n, int nact, int D, int32_t H, int64_t hi,
                                           const int64_t *arrival, const int32_t *ids,
                                           const int32_t *cch, const int32_t *Uq,
                                           int32_t *choice_out, uint8_t *st, int32_t *dec,
                                           long long *disp, int32_t *g, int32_t *U, int32_t *act,
                                           StreamState *S, int32_t *status) {
  pdl_prologue();
  const long long s = arrival[hi - 1];
  const int stride = gridDim.x * blockDim.x;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const int id = ids[i];
    int c = cch ? cch[i] : id % D;
    if (c < 0 || c >= D) {  // only after a range error (a bound that overflowed)
      flag_error(status, MAPS_E_RANGE);
      c = 0;
    }
    choice_out[id] = c;
    st[id] = kWaiting;
    dec[id] = c;
    disp[id] = s;
    g[id] = 0;
    U[id] = cch ? Uq[nact + i] : H;
    act[nact + i] = id;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) S->nact = nact + n;
}

// 6. The batch joins the waiting queues of its decoders.
__global__ void stream_enqueue_kernel(int64_t lo, int nb, int nact, int64_t hi, int D,
                                      const int64_t *arrival, const int32_t *choice,
                                      const int32_t *Uq, uint8_t *st, int32_t *dec,
                                      long long *disp, int32_t *g, int32_t *U, int32_t *act,
                                      StreamState *S, int32_t *status) {
  pdl_prologue();
  const long long s = arrival[hi - 1];
  const int stride = gridDim.x * blockDim.x;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nb; i += stride) {
    const int64_t id = lo + i;
    int c = choice[id];
    if (c < 0 || c >= D) {  // only after a range error (a bound that overflowed)
      flag_error(status, MAPS_E_RANGE);
      c = 0;
    }
    st[id] = kWaiting;
    dec[id] = c;
    disp[id] = s;
    g[id] = 0;
    U[id] = Uq[nact + i];
    act[nact + i] = static_cast<int32_t>(id);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) S->nact = nact + nb;
}

// 7. The waiting requests with their order keys.
__global__ void __launch_bounds__(kSt, 1)
stream_waitlist_kernel(int n, int64_t hi, const int64_t *arrival, const int32_t *act,
                       const uint8_t *st, const int32_t *dec, const int32_t *U,
                       const long long *disp, int32_t *wid, int32_t *wdec, int32_t *wU,
                       int32_t *wwait, int32_t *warr) {
  pdl_prologue();
  __shared__ int s_w[kStWarps];
  const long long s = arrival[hi - 1];
  int nw = 0;
  for (int c0 = 0; c0 < n; c0 += kSt) {
    const int x = c0 + threadIdx.x;
    const int id = x < n ? act[x] : -1;
    const bool f = id >= 0 && st[id] == kWaiting;
    int tot;
    const int pos = block_flag_scan(f, s_w, tot);
    if (f) {
      const int o = nw + pos;
      const long long w = s - disp[id];
      wid[o] = id;
      wdec[o] = dec[id];
      wU[o] = U[id];
      wwait[o] = static_cast<int32_t>(w > 0x7fffffffLL ? 0x7fffffffLL : w);
      warr[o] = id;
    }
    nw += tot;
  }
}

// 8. Admission, one warp per decoder: entry x of the queue is admitted while
//    it and every entry before it satisfy used + (the increments of the
//    entries admitted before) + p + U <= cap, the increment being p, p + U
//    (staged) or 2p + U (held).  Each decoder's statistics gain its queue
//    left waiting times the steps to the next batch, and its admissions.
__global__ void __launch_bounds__(kSt, 1)
//    Per-step mode: each admission's sequence number (aseq), the queue's
//    first entry left (qhead), and the waiting requests count for the
//    dispatch step alone (the steps after it are the next interval's).
stream_admit_kernel(int D, int32_t cap, int acct, int per_step, int nw, int64_t hi, int64_t hi_next,
                    const int64_t *arrival, const int64_t *wseg, const int32_t *wperm,
                    const int32_t *wid, const int32_t *prompt, const int32_t *U,
                    const long long *used, uint8_t *st, int32_t *g, int32_t *res_u,
                    long long *aseq, long long *dseq, int64_t *qhead, const StreamState *S,
                    int64_t *stats_b, int64_t *dst) {
  pdl_prologue();
  __shared__ int s_adm;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const long long span = per_step ? (hi_next != hi ? 1 : 0) : arrival[hi_next - 1] - arrival[hi - 1];
  if (tid == 0) s_adm = 0;
  __syncthreads();
  for (int k = warp; k < D; k += kStWarps) {
    long long u = used[k];
    const long long x1 = wseg[k + 1];
    int adm = 0;
    bool stop = false;
    for (long long b0 = wseg[k]; b0 < x1 && !stop; b0 += 32) {
      const long long x = b0 + lane;
      const bool valid = x < x1;
      const int id = valid ? wid[wperm[x]] : -1;
      const long long p = valid ? prompt[id] : 0, uu = valid ? U[id] : 0;
      const long long inc = acct == MAPS_STREAM_OCCUPANCY ? p
                            : acct == MAPS_STREAM_STAGED  ? p + uu
                                                          : 2 * p + uu;
      long long incl = inc;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      const bool ok = valid && u + (incl - inc) + p + uu <= cap;
      const unsigned fail = __ballot_sync(0xffffffffu, valid && !ok);
      const unsigned vmask = __ballot_sync(0xffffffffu, valid);
      const int nadm = fail ? __ffs(fail) - 1 : __popc(vmask);
      if (lane < nadm) {
        st[id] = kRunning;
        g[id] = 0;
        res_u[id] = static_cast<int32_t>(uu);
        if (per_step) aseq[id] = dseq[k] + adm + lane;
      }
      if (nadm > 0) u += __shfl_sync(0xffffffffu, incl, nadm - 1);
      adm += nadm;
      stop = fail != 0;
    }
    if (lane == 0 && adm) atomicAdd(&s_adm, adm);
    if (lane == 0) {  // decoder k is this warp's alone
      if (per_step) {
        dseq[k] += adm;
        qhead[k] = wseg[k] + adm;
      }
      if (dst != nullptr) {
        dst[4 * k] += (x1 - wseg[k] - adm) * span;
        dst[4 * k + 2] += adm;
      }
    }
  }
  __syncthreads();
  if (tid == 0) {
    stats_b[1] = s_adm + (per_step ? S->adm_i : 0);
    stats_b[2] = nw - s_adm;
  }
}

struct StreamWs {
  size_t sub_bytes;  // [0, sub_bytes): workspace of the calls the loop makes
  StreamState *S;
  uint8_t *st;
  int32_t *g, *dec, *U, *res_u;
  long long *disp;
  int32_t *act[2];
  int32_t *done_id, *done_rem, *done_perm, *zeros;
  int64_t *done_seg;
  int32_t *win_true, *win_pred, *qpred, *Uq;
  int64_t *res_off;
  int32_t *rp, *rg, *rU, *capv, *Q;
  long long *used;
  int32_t *K;
  int64_t *headroom;
  int32_t *wid, *wdec, *wU, *wwait, *warr, *wperm;
  int64_t *wseg;
  int32_t *q_dev;
  // deferral
  int32_t *pend[2], *cid, *tout, *cp, *cch;
  // per-step mode
  long long *aseq, *dseq;
  int32_t *rbuf, *sbuf;
  int64_t *qhead;
};

size_t stream_sub_bytes(const maps_stream_cfg &c) {
  size_t b = maps_calibrate_workspace_size(c.window, c.N);
  b = std::max(b, maps_project_occupancy_workspace_size(c.D, c.H, c.N));
  b = std::max(b, maps_dispatch_workspace_size(MAPS_MODE_SEQUENTIAL, c.D, c.H, c.batch));
  b = std::max(b, maps_order_local_workspace_size(c.N, c.D));
  b = std::max(b, maps_order_local_workspace_size(c.N, 1));
  return (b + kAlign - 1) / kAlign * kAlign;
}

StreamWs carve_stream(Carve &c, const maps_stream_cfg &cfg) {
  StreamWs w;
  const size_t N = static_cast<size_t>(cfg.N), D = static_cast<size_t>(cfg.D);
  w.sub_bytes = stream_sub_bytes(cfg);
  c.off = w.sub_bytes;
  w.S = c.take<StreamState>(1);
  w.st = c.take<uint8_t>(N);
  w.g = c.take<int32_t>(N);
  w.dec = c.take<int32_t>(N);
  w.U = c.take<int32_t>(N);
  w.res_u = c.take<int32_t>(N);
  w.disp = c.take<long long>(N);
  w.act[0] = c.take<int32_t>(N);
  w.act[1] = c.take<int32_t>(N);
  w.done_id = c.take<int32_t>(N);
  w.done_rem = c.take<int32_t>(N);
  w.done_perm = c.take<int32_t>(N);
  w.zeros = c.take<int32_t>(N);
  w.done_seg = c.take<int64_t>(2);
  w.win_true = c.take<int32_t>(static_cast<size_t>(cfg.window));
  w.win_pred = c.take<int32_t>(static_cast<size_t>(cfg.window));
  w.qpred = c.take<int32_t>(N);
  w.Uq = c.take<int32_t>(N);
  w.res_off = c.take<int64_t>(D + 1);
  w.rp = c.take<int32_t>(N);
  w.rg = c.take<int32_t>(N);
  w.rU = c.take<int32_t>(N);
  w.capv = c.take<int32_t>(D);
  w.Q = c.take<int32_t>(D);
  w.used = c.take<long long>(D);
  w.K = c.take<int32_t>(D * static_cast<size_t>(cfg.H));
  w.headroom = c.take<int64_t>(static_cast<size_t>(cfg.batch));
  w.wid = c.take<int32_t>(N);
  w.wdec = c.take<int32_t>(N);
  w.wU = c.take<int32_t>(N);
  w.wwait = c.take<int32_t>(N);
  w.warr = c.take<int32_t>(N);
  w.wperm = c.take<int32_t>(N);
  w.wseg = c.take<int64_t>(D + 1);
  w.q_dev = c.take<int32_t>(1);
  const bool defer = cfg.beta >= 0;
  w.pend[0] = c.take<int32_t>(defer ? N : 0);
  w.pend[1] = c.take<int32_t>(defer ? N : 0);
  w.cid = c.take<int32_t>(defer ? N : 0);
  w.tout = c.take<int32_t>(defer ? N : 0);
  w.cp = c.take<int32_t>(defer ? N : 0);
  w.cch = c.take<int32_t>(defer ? N : 0);
  const bool ps = cfg.per_step != 0;
  w.aseq = c.take<long long>(ps ? N : 0);
  w.dseq = c.take<long long>(ps ? D : 0);
  w.rbuf = c.take<int32_t>(ps ? N : 0);
  w.sbuf = c.take<int32_t>(ps ? N : 0);
  w.qhead = c.take<int64_t>(ps ? D : 0);
  return w;
}

bool cfg_ok(const maps_stream_cfg *c) {
  return c != nullptr && c->N >= 1 && c->N <= 0x7fffffffLL && c->D >= 1 && c->D <= kStreamMaxD &&
         c->H >= 1 && c->H <= (1 << 28) && c->cap >= 0 && c->batch >= 1 && c->window >= 1 &&
         c->alpha_ppm > 0 && c->alpha_ppm < 1000000u && c->dispatch_policy >= MAPS_STREAM_MAPS &&
         c->dispatch_policy <= MAPS_STREAM_LR && c->local_order >= MAPS_STREAM_SJF &&
         c->local_order <= MAPS_STREAM_FCFS && c->accounting >= MAPS_STREAM_OCCUPANCY &&
         c->accounting <= MAPS_STREAM_HELD && (c->per_step == 0 || c->per_step == 1);
}

int grid_for(int64_t n, int threads = 256) {
  return static_cast<int>(std::max<int64_t>(1, std::min<int64_t>((n + threads - 1) / threads,
                                                                 4LL * sm_count())));
}

}  // namespace
}  // namespace maps

extern "C" {

size_t maps_stream_workspace_size(const maps_stream_cfg *cfg) {
  using namespace maps;
  if (!cfg_ok(cfg)) return kCtrlBytes;
  Carve c(nullptr);
  carve_stream(c, *cfg);
  return c.bytes();
}

int maps_stream_run(const maps_stream_cfg *cfg, const int64_t *arrival_ms, const int32_t *prompt,
                    const int32_t *true_len, const int32_t *pred, const int32_t *pred_delay,
                    int32_t *choice_out, int32_t *q_out, int64_t *stats_out,
                    int64_t *dec_stats_out, void *ws, size_t ws_bytes, void *stream) {
  using namespace maps;
  if (!cfg_ok(cfg) || arrival_ms == nullptr || prompt == nullptr || true_len == nullptr ||
      pred == nullptr || choice_out == nullptr || q_out == nullptr || stats_out == nullptr ||
      (cfg->beta >= 0 && pred_delay == nullptr))
    return MAPS_E_INVALID;
  MAPS_TRY(check_ws(ws, ws_bytes, maps_stream_workspace_size(cfg)));
  const maps_stream_cfg c = *cfg;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t *status = status_word(ws);
  Carve cv(ws);
  const StreamWs w = carve_stream(cv, c);
  const int64_t N = c.N, B = c.batch, nbatch = (N + B - 1) / B;
  const int D = c.D;
  const bool defer = c.beta >= 0;
  const int per_step = c.per_step;
  const int32_t *pdl = defer ? pred_delay : nullptr;

  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.st, 0, static_cast<size_t>(N), s)));
  MAPS_TRY(cuda_ok(cudaMemsetAsync(w.zeros, 0, static_cast<size_t>(N) * sizeof(int32_t), s)));
  if (dec_stats_out != nullptr)
    MAPS_TRY(cuda_ok(cudaMemsetAsync(dec_stats_out, 0, static_cast<size_t>(c.D) * 4 * sizeof(int64_t), s)));
  if (per_step) {
    MAPS_TRY(cuda_ok(cudaMemsetAsync(w.dseq, 0, static_cast<size_t>(D) * sizeof(long long), s)));
    MAPS_TRY(cuda_ok(cudaMemsetAsync(w.qhead, 0, static_cast<size_t>(D) * sizeof(int64_t), s)));
    MAPS_TRY(cuda_ok(cudaMemsetAsync(w.wseg, 0, static_cast<size_t>(D + 1) * sizeof(int64_t), s)));
  }
  launch_pdl(stream_init_kernel, 1, kSt, 0, s, std::min(N, B), D, c.cap, arrival_ms, w.capv, w.S);
  launch_pdl(stream_validate_kernel, grid_for(N), 256, 0, s, N, arrival_ms, prompt, true_len, pred,
             pdl, status);
  MAPS_TRY(launch_ok());
  {
    const int st0 = maps_check(ws, stream);  // a bad input stops the loop before it starts
    if (st0 != MAPS_OK) return st0;
  }

  long long total_done = 0;
  StreamState hs;
  for (int64_t b = 0; b < nbatch; ++b) {
    const int64_t lo = b * B, hi = std::min(lo + B, N);
    const int nb = static_cast<int>(hi - lo);
    int32_t *act_in = w.act[b & 1], *act = w.act[(b & 1) ^ 1];
    int64_t *stats_b = stats_out + 4 * b;
    if (defer)  // 4 (first half): who is dispatched at this step
      launch_pdl(stream_select_kernel, 1, kSt, 0, s, lo, nb, hi, c.beta, b + 1 == nbatch ? 1 : 0,
                 arrival_ms, pred_delay, w.pend[b & 1], w.pend[(b & 1) ^ 1], w.cid, w.tout, w.S);
    if (per_step)  // 1'.
      launch_pdl(stream_interval_kernel, 1, kSt, 0, s, hi, D, c.cap, c.accounting, arrival_ms,
                 prompt, true_len, w.U, w.res_u, w.st, w.g, w.dec, act_in, w.wid, w.wperm, w.wseg,
                 w.qhead, w.aseq, w.dseq, w.rbuf, w.sbuf, w.done_id, w.done_rem, w.S, dec_stats_out);
    launch_pdl(stream_advance_kernel, 1, kSt, 0, s, hi, D, c.cap, c.accounting, per_step, arrival_ms,
               prompt, true_len, w.res_u, w.st, w.g, w.dec, act_in, act, w.done_id, w.done_rem,
               w.used, w.S, stats_b, dec_stats_out);
    MAPS_TRY(launch_ok());
    MAPS_TRY(cuda_ok(cudaMemcpyAsync(&hs, w.S, sizeof(hs), cudaMemcpyDeviceToHost, s)));
    MAPS_TRY(cuda_ok(cudaStreamSynchronize(s)));
    int nact = hs.nact;
    const int ndone = hs.ndone, nwait = hs.nwait;
    // the policy's candidates: the batch, or (deferral) the listed ids
    const int nc = defer ? hs.nc : nb, nto = defer ? hs.nto : 0;
    const int32_t *cids = defer ? w.cid : nullptr;
    const int32_t *cpr = defer ? w.cp : prompt + lo;
    int32_t *cch = defer ? w.cch : choice_out + lo;

    if (ndone > 0) {  // 2.
      MAPS_TRY(maps_order_local(ndone, 1, w.zeros, w.done_rem, w.zeros, w.done_id, 0, w.done_perm,
                                w.done_seg, ws, w.sub_bytes, stream));
      launch_pdl(stream_window_kernel, grid_for(ndone), 256, 0, s, ndone, total_done, c.window,
                                                           w.done_perm, w.done_id, true_len, pred,
                                                           w.win_true, w.win_pred);
      total_done += ndone;
    }
    const int64_t win_len = std::min<long long>(total_done, c.window);
    if (nto > 0) {  // 4 (second half): timed out, round robin with the horizon as bound
      launch_pdl(stream_enqueue_list_kernel, grid_for(nto), 256, 0, s, nto, nact, D, c.H, hi,
                 arrival_ms, w.tout, nullptr, w.Uq, choice_out, w.st, w.dec, w.disp, w.g, w.U, act,
                 w.S, status);
      nact += nto;
    }

    launch_pdl(stream_gather_kernel, grid_for(nact + nc), 256, 0, s, nact, nc, lo, act, cids, pred,
               prompt, w.qpred, w.cp);
    const int cs = maps_calibrate(w.win_true, w.win_pred, win_len, c.alpha_ppm, w.qpred, nact + nc,
                                  w.Uq, w.q_dev, nullptr, ws, w.sub_bytes, stream);  // 3.
    const bool rr = cs == MAPS_E_UNBOUNDED;
    if (cs != MAPS_OK && !rr) return cs;
    if (rr)
      launch_pdl(stream_rr_kernel, grid_for(nact + nc), 256, 0, s, nact + nc, nc, lo, D, 1, w.qpred,
                 w.Uq, cids, cch);
    launch_pdl(stream_csr_kernel, 1, kSt, 0, s, nact, D, rr ? 1 : 0, w.q_dev, q_out + b, act, w.st, w.g,
               w.dec, prompt, w.Uq, w.U, w.res_off, w.rp, w.rg, w.rU, w.Q, arrival_ms, pdl, hi,
               c.H);  // 4.
    MAPS_TRY(launch_ok());
    const int mc = c.dispatch_policy == MAPS_STREAM_MC ? 1 : 0;
    if (nc == 0) {
      // nobody to dispatch at this step
    } else if (!rr && c.dispatch_policy == MAPS_STREAM_RR) {  // 5'.
      launch_pdl(stream_rr_kernel, grid_for(nc), 256, 0, s, nc, nc, lo, D, 0, w.qpred, w.Uq, cids, cch);
      MAPS_TRY(launch_ok());
    } else if (!rr && c.dispatch_policy == MAPS_STREAM_LR) {
      launch_pdl(stream_lr_kernel, 1, 32, 0, s, D, nc, w.res_off, cch);
      MAPS_TRY(launch_ok());
    } else if (!rr) {  // 5.
      const size_t dsm = stream_dispatch_smem(D, nact, nc);
      if (dsm + 2048 <= static_cast<size_t>(max_smem_optin())) {
        // the decoders' pairs fit in shared memory: no dense projection
        MAPS_TRY(cuda_ok(cudaFuncSetAttribute(stream_dispatch_kernel,
                                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(dsm))));
        launch_pdl(stream_dispatch_kernel, 1, kSt, dsm, s, D, c.H, nc, mc, w.res_off, w.rp, w.rg,
                   w.rU, w.capv, w.Q, cpr, w.Uq + nact, cch, nullptr, status);  // no headroom out
        MAPS_TRY(launch_ok());
      } else {
        MAPS_TRY(maps_project_occupancy(D, c.H, w.res_off, nact, w.rp, w.rg, w.rU, w.K, nullptr, ws,
                                        w.sub_bytes, stream));
        MAPS_TRY(dispatch_sequential(D, c.H, w.K, w.capv, w.Q, nc, cpr, w.Uq + nact, cch,
                                     w.headroom, mc != 0, ws, s));
      }
    }
    if (defer) {
      if (nc > 0)
        launch_pdl(stream_enqueue_list_kernel, grid_for(nc), 256, 0, s, nc, nact, D, c.H, hi,
                   arrival_ms, w.cid, w.cch, w.Uq, choice_out, w.st, w.dec, w.disp, w.g, w.U, act,
                   w.S, status);  // 6.
    } else {
      launch_pdl(stream_enqueue_kernel, grid_for(nb), 256, 0, s, lo, nb, nact, hi, D, arrival_ms,
                 choice_out, w.Uq, w.st, w.dec, w.disp, w.g, w.U, act, w.S, status);  // 6.
    }
    const int n_all = nact + nc, nw = nwait + nto + nc;
    launch_pdl(stream_waitlist_kernel, 1, kSt, 0, s, n_all, hi, arrival_ms, act, w.st, w.dec, w.U, w.disp,
                                             w.wid, w.wdec, w.wU, w.wwait, w.warr);  // 7.
    MAPS_TRY(launch_ok());
    // FCFS: every wait is >= 0 > -1, so every entry is promoted: arrival order
    const int32_t mw = c.local_order == MAPS_STREAM_FCFS ? -1 : c.max_wait;
    MAPS_TRY(maps_order_local(nw, D, w.wdec, w.wU, w.wwait, w.warr, mw, w.wperm, w.wseg, ws,
                              w.sub_bytes, stream));
    const int64_t hi_next = b + 1 < nbatch ? std::min(hi + B, N) : hi;
    launch_pdl(stream_admit_kernel, 1, kSt, 0, s, D, c.cap, c.accounting, per_step, nw, hi, hi_next,
               arrival_ms, w.wseg, w.wperm, w.wid, prompt, w.U, w.used, w.st, w.g, w.res_u, w.aseq,
               w.dseq, w.qhead, w.S, stats_b, dec_stats_out);  // 8.
    MAPS_TRY(launch_ok());
  }
  return maps_check(ws, stream);
}

}  // extern "C"
