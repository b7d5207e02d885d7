/*
 * maps.h -- C ABI of the MAPS memory-aware predictive scheduler hot path,
 * implemented as integer-only CUDA kernels for GB300 (sm_103a).
 *
 * The four calls follow the scheduler's problem statement (Sec. 3.3): decoders
 * d_k with KV-token capacity C_k and waiting-queue length Q_k; requests with a
 * prompt length, a predicted output length, and a calibrated upper bound on
 * it (Sec. 3.2).
 *
 * Conventions shared by every call
 * --------------------------------
 * Memory.   Every array argument is DEVICE memory owned by the caller, except
 *           where an argument name ends in `_host`.  The library allocates
 *           nothing: calls that need scratch memory take a caller-provided
 *           workspace `ws` of `ws_bytes` bytes, sized by the matching
 *           `maps_*_workspace_size()` query.  A workspace must be zero-filled
 *           before its first use and must be 256-byte aligned.  One
 *           workspace may serve several calls in sequence on one stream;
 *           calls that run concurrently need separate workspaces.
 * Streams.  `stream` is a cudaStream_t passed as void*.  Calls enqueue work
 *           on it and return without waiting, except where a `_host` output
 *           is non-NULL: then the call synchronises the stream and returns
 *           the full status, data-dependent errors included.
 * Grids.    maps_calibrate with more than 8,192 residuals and
 *           maps_order_local past one block each launch one cooperative
 *           kernel (every block resident at once, with bounded grid
 *           barriers): such a launch starts when the multiprocessors it
 *           needs are free, so it waits for other streams' kernels that hold
 *           them.
 * Layout.   Arrays are dense and row-major; int32 unless stated.  K is
 *           [D][H].  Residents of decoder k are the index range
 *           [res_off[k], res_off[k+1]) of the resident arrays (CSR).
 * Status.   Every call returns an int status.  Argument errors (NULL
 *           pointers, negative sizes, a workspace too small or misaligned)
 *           are returned at once and nothing is enqueued.  Errors that depend
 *           on device data (a value outside its domain, an int32 overflow, a
 *           bounded device wait that expired) are recorded in a sticky status
 *           word inside the workspace; read and clear it with maps_check().
 *           Outputs are unspecified when a call or a later maps_check()
 *           reports an error.  No exception crosses the interface and no
 *           kernel traps.
 * Domain.   Lengths (prompt p, generated g, bounds U), capacities, queue
 *           lengths and K values must be >= 0; a negative one is reported as
 *           MAPS_E_RANGE.
 * Aliasing. An output array overlaps no input array, no other output and no
 *           workspace of the same call.
 */
#ifndef MAPS_H
#define MAPS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MAPS_OK 0
#define MAPS_E_INVALID (-1)   /* bad argument: NULL, size, alignment, mode */
#define MAPS_E_RANGE (-2)     /* device data outside its domain or int32 range */
#define MAPS_E_UNBOUNDED (-3) /* conformal rank exceeds n: no finite bound */
#define MAPS_E_TIMEOUT (-4)   /* a bounded device wait expired */
#define MAPS_E_CUDA (-5)      /* CUDA runtime error; see maps_last_cuda_error */
#define MAPS_E_WORKSPACE (-6) /* workspace smaller than the size query asked */

#define MAPS_MODE_SNAPSHOT 0
#define MAPS_MODE_SEQUENTIAL 1
#define MAPS_MODE_ALG1_SNAPSHOT 2
#define MAPS_MODE_ALG1_SEQUENTIAL 3

/* Library version, major*10000 + minor*100 + patch. */
int maps_version(void);

/* The cudaError_t behind the last MAPS_E_CUDA returned by this thread. */
int maps_last_cuda_error(void);

/* Synchronises `stream`, returns the workspace's sticky device status
 * (MAPS_OK or the first error any kernel recorded in it) and clears it. */
int maps_check(void *ws, void *stream);

/* ------------------------------------------------------------------------
 * Uncertainty-aware calibration, Sec. 3.2.
 *
 * Scores s_i = max(0, true_len[i] - pred_len[i]) (Eq. nonconformity) over the
 * calibration set of n completed requests; q = the k-th smallest score with
 * k = ceil((1 - alpha)(n + 1)), alpha = alpha_ppm / 1e6 (the rank is exact
 * integer arithmetic); then, for m query predictions, the calibrated upper
 * bounds bound_out[i] = query_pred[i] + q (Eq. conformal_upper).
 *
 *   true_len, pred_len  [n] int32, device.
 *   alpha_ppm           miscoverage in parts per million, 0 < alpha_ppm < 1e6.
 *   query_pred, m       [m] predictions to bound (m may be 0, then both NULL).
 *   bound_out           [m] int32 output, device.
 *   q_dev_out           int32 scalar output, device (may be NULL).
 *   q_host_out          int32 scalar output, host (may be NULL; non-NULL
 *                       synchronises the stream).
 * Returns MAPS_E_UNBOUNDED at once, enqueuing nothing, when k > n (including
 * n = 0): the bound is unavailable and Alg. 1 falls back to round robin.
 * q > INT32_MAX or a bound above INT32_MAX is MAPS_E_RANGE.
 * Requires n <= 2^40.
 * ---------------------------------------------------------------------- */
size_t maps_calibrate_workspace_size(int64_t n, int64_t m);
int maps_calibrate(const int32_t *true_len, const int32_t *pred_len, int64_t n,
                   uint32_t alpha_ppm, const int32_t *query_pred, int64_t m,
                   int32_t *bound_out, int32_t *q_dev_out, int32_t *q_host_out,
                   void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * Projected KV-token occupancy over a step horizon.
 *
 * Built on the KV footprint M(r) = L_p + L_out (App. A, Eq. kv_demand) and the
 * occupancy K_d(t) of Eq. (admission): at step t in [0, H) a resident r of
 * decoder k with prompt p, g tokens generated and bound U holds p + g + t + 1
 * KV tokens while t < e_r = min(max(U - g, 1), H) (a resident past its bound
 * is kept for one step), so
 *     K[k][t] = sum over residents r of k with t < e_r of (p + g + 1 + t).
 *
 *   D, H                decoders (>= 1) and horizon steps (1 <= H <= 2^28;
 *                       a larger H is MAPS_E_INVALID).
 *   res_off             [D+1] int64 CSR offsets into the resident arrays,
 *                       non-decreasing within [0, R].
 *   R                   length of prompt / gen / bound.
 *   prompt, gen, bound  [R] int32 resident prompt lengths, generated tokens,
 *                       calibrated bounds.
 *   K_out               [D][H] int32 output.
 *   kmax_out            optional [D][ceil(H/16)] uint32 output (NULL: not
 *                       written): kmax[k][b] = max over the steps t of block
 *                       b (t in [16b, min(16b+16, H))) of K[k][t] + t.  It
 *                       summarises K for maps_dispatch (SNAPSHOT), which
 *                       then need not re-read the whole of K.
 * A K value above INT32_MAX, offsets out of order or a negative length is
 * MAPS_E_RANGE (via maps_check).
 * ---------------------------------------------------------------------- */
size_t maps_project_occupancy_workspace_size(int32_t D, int32_t H, int64_t R);
int maps_project_occupancy(int32_t D, int32_t H, const int64_t *res_off,
                           int64_t R, const int32_t *prompt, const int32_t *gen,
                           const int32_t *bound, int32_t *K_out,
                           uint32_t *kmax_out, void *ws, size_t ws_bytes,
                           void *stream);

/* ------------------------------------------------------------------------
 * Global memory-aware dispatch, Sec. 3.3 and Alg. 1.
 *
 * Horizon modes (SNAPSHOT, SEQUENTIAL).  Candidate j (prompt p_j, bound U_j)
 * is live for u_j = min(max(U_j, 1), H) steps holding p_j + t + 1 tokens, so
 * on decoder k its peak is
 *     peak_jk = max_{t < u_j} (K[k][t] + p_j + t + 1),  h_jk = cap[k] - peak_jk.
 * Decoder k is feasible iff h_jk >= 0.  The choice is the feasible decoder
 * with the smallest Q[k]; if none is feasible, the decoder with the largest
 * headroom h_jk (the fallback to the most available capacity).  Ties go to
 * the lowest decoder index.  SNAPSHOT scores every candidate against the same
 * state.  SEQUENTIAL takes candidates in index order and, after each choice,
 * reserves the footprint at the chosen decoder: K[k*][t] += p_j + t + 1 for
 * t < u_j and Q[k*] += 1, in place.
 *
 * ALG1 modes (ALG1_SNAPSHOT, ALG1_SEQUENTIAL): Algorithm 1 literally, with
 * block size S: B_need_j = ceil((p_j + U_j) / S) (Eq. feasibility);
 * B_eff_k = floor(cap[k] / S) - sum over residents of
 * ceil((p + max(U, g + 1)) / S) (free blocks minus what each ongoing request
 * holds or has reserved at its bound); feasible iff B_need_j <= B_eff_k; argmin
 * Q over the feasible set, else argmax B_eff; headroom = B_eff - B_need.
 * ALG1_SEQUENTIAL subtracts B_need from B_eff[k*] and adds 1 to Q[k*] after
 * each choice.  K is not read in the ALG1 modes.
 *
 *   mode                MAPS_MODE_*.
 *   D, H, S             decoders (1 <= D <= 1024), horizon (1 <= H <= 2^28),
 *                       block size (ALG1).
 *   K                   [D][H] int32 occupancy (horizon modes; updated in
 *                       place by SEQUENTIAL).
 *   kmax                optional [D][ceil(H/16)] uint32, SNAPSHOT only: the
 *                       summary maps_project_occupancy wrote for this same K.
 *                       NULL makes the call derive it from K (one more pass
 *                       over K).  The call compares a given summary with K at
 *                       four blocks of every row and reports a mismatch there
 *                       as MAPS_E_INVALID (via maps_check); a summary that
 *                       differs from K elsewhere gives unspecified results.
 *   cap, Q              [D] int32 capacities and queue lengths (Q updated in
 *                       place by the SEQUENTIAL modes).
 *   res_off, R, prompt, gen, bound   residents as in maps_project_occupancy
 *                       (ALG1 modes only; else NULL / 0).
 *   J                   number of candidates.
 *   cand_prompt, cand_bound   [J] int32.
 *   choice_out          [J] int32 output decoder index.
 *   headroom_out        [J] int64 output headroom at the chosen decoder
 *                       (tokens, or blocks in ALG1 modes); may be NULL.
 * ---------------------------------------------------------------------- */
size_t maps_dispatch_workspace_size(int32_t mode, int32_t D, int32_t H,
                                    int64_t J);

int maps_dispatch(int32_t mode, int32_t D, int32_t H, int32_t S, int32_t *K,
                  const uint32_t *kmax, const int32_t *cap, int32_t *Q,
                  const int64_t *res_off,
                  int64_t R, const int32_t *prompt, const int32_t *gen,
                  const int32_t *bound, int64_t J, const int32_t *cand_prompt,
                  const int32_t *cand_bound, int32_t *choice_out,
                  int64_t *headroom_out, void *ws, size_t ws_bytes,
                  void *stream);

/* ------------------------------------------------------------------------
 * Local SJF reordering, Sec. 3.3: Order(Q_k) = argsort of the calibrated
 * bound, with the maximum-waiting-time promotion.
 *
 * Entries are grouped by decoder; within a decoder, entries with
 * wait > max_wait come first in arrival order, then the rest by ascending
 * bound, ties by arrival, then by entry index.
 *
 *   N, D                entries (N <= INT32_MAX) and decoders (>= 1).
 *   dec                 [N] int32 decoder of each entry, in [0, D).
 *   bound               [N] int32 calibrated bound (>= 0).
 *   wait                [N] int32 steps waited so far.
 *   arrival             [N] int32 arrival index (>= 0).
 *   max_wait            promotion threshold in steps.
 *   perm_out            [N] int32 output: entry indices in queue order.
 *   seg_off_out         [D+1] int64 output: decoder k's entries are
 *                       perm_out[seg_off_out[k] .. seg_off_out[k+1]).
 * ---------------------------------------------------------------------- */
size_t maps_order_local_workspace_size(int64_t N, int32_t D);
int maps_order_local(int64_t N, int32_t D, const int32_t *dec,
                     const int32_t *bound, const int32_t *wait,
                     const int32_t *arrival, int32_t max_wait,
                     int32_t *perm_out, int64_t *seg_off_out, void *ws,
                     size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------
 * maps_order_local without any allocation.  The paper has no counterpart:
 * this is a deployment aid.
 *
 * Some callers cannot call cudaMalloc at all -- for instance a scheduler
 * embedded in a host process whose device allocator belongs to another
 * framework, or one that must not allocate once it is serving.  This call
 * computes exactly what maps_order_local computes, but its scratch memory is
 * a fixed array of 5 MiB compiled into the library (every GPU that loads the
 * library holds it until the process exits), so it takes no workspace and
 * allocates nothing.  The caller still provides inputs and outputs, in
 * device memory, as for maps_order_local.
 *
 *   Limits              N <= 65,536 entries and D <= 4,096 decoders; larger
 *                       sizes return MAPS_E_WORKSPACE at once.
 *   status_host         optional host int32 (NULL: not written).  Non-NULL
 *                       synchronises the stream and returns the full status,
 *                       data-dependent errors included.  With NULL, data
 *                       errors (MAPS_E_RANGE, MAPS_E_TIMEOUT) are lost: the
 *                       array's status word is cleared by the next call and
 *                       no other call reads it, so a caller that needs them
 *                       must pass status_host.
 *   First call          every call looks up the array's device address on
 *                       the current device (a host call); the first call on a
 *                       device may also load the library's device code there,
 *                       so make that first call before any stream capture.
 *   Concurrency         every call shares the one array: calls whose work
 *                       overlaps on the GPU (other streams, other threads)
 *                       race and give wrong results.  Order them on one
 *                       stream.
 * ---------------------------------------------------------------------- */
int maps_order_local_static(int64_t N, int32_t D, const int32_t *dec,
                            const int32_t *bound, const int32_t *wait,
                            const int32_t *arrival, int32_t max_wait,
                            int32_t *perm_out, int64_t *seg_off_out,
                            int32_t *status_host, void *stream);

/* ------------------------------------------------------------------------
 * The streaming scheduler loop, run on the device end to end.
 *
 * Requests arrive with arrival step arrival_ms[i] (1 ms per decode step,
 * non-decreasing in i) and are dispatched in batches of cfg->batch in index
 * order; batch b is dispatched at the arrival step s_b of its last request.
 * Per batch, following Sec. 3.2 (sliding calibration window), Sec. 3.3
 * (memory-aware dispatch, local SJF order with promotion), Algorithm 1 (round
 * robin when no bound is available) and App. A Eq. (admission):
 *   1. every running request generates s_b - s_{b-1} tokens (one per step);
 *      one that reaches its true length completes at the step it does;
 *   2. completions enter a window of the last cfg->window completed
 *      requests, ordered by (completion step, index);
 *   3. q = the conformal quantile of the window (maps_calibrate); every
 *      request in the system and in the batch gets U = pred + q.  If the
 *      quantile is unbounded (too few completions) U = pred, q_out[b] = -1
 *      and the batch is dispatched round robin: choice = index mod D;
 *   4. otherwise occupancy is projected over the running (g generated) and
 *      waiting (g = 0) requests and the batch is dispatched SEQUENTIALly
 *      (maps_dispatch) with Q[k] = requests waiting at decoder k;
 *   5. the batch joins the chosen decoders' waiting queues;
 *   6. each waiting queue is put in local order (maps_order_local, with
 *      wait = s_b - dispatch step) and admitted in that order while
 *      used + p + U <= cap (used = prompt + generated tokens of the running
 *      requests, grown by p per admission); the first misfit stops its queue.
 * No preemption; a running request above capacity is only counted.
 *
 * Policy variants (the Sec. 4 ablations and the baselines of the App. C
 * studies), chosen in cfg; the defaults (all 0) are the loop above:
 *   dispatch_policy  MAPS_STREAM_MAPS: SEQUENTIAL dispatch as in 4;
 *                    MAPS_STREAM_MC: the same projection, every candidate to
 *                    the decoder of largest headroom cap - (p + 1 + M), ties
 *                    to the lowest index (memory-only, no queue term);
 *                    MAPS_STREAM_RR: round robin, choice = index mod D;
 *                    MAPS_STREAM_LR: least requests, the decoder with the
 *                    fewest requests in the system (running and waiting),
 *                    the batch counted as it is dispatched, ties to the
 *                    lowest index.  An unbounded quantile still sends the
 *                    batch round robin under every policy.
 *   local_order      MAPS_STREAM_SJF: as in 6; MAPS_STREAM_FCFS: every queue
 *                    in arrival (index) order.
 *   accounting       what a running request counts for in `used`, with
 *                    g generated and U* its bound at admission:
 *                    MAPS_STREAM_OCCUPANCY  p + g (grown by p per admission);
 *                    MAPS_STREAM_STAGED     p + max(U*, g) (the output stays
 *                      reserved at its bound; grown by p + U);
 *                    MAPS_STREAM_HELD       2p + max(U*, g) (the prompt is
 *                      held twice, at the prefill and decode sides, as when
 *                      the staged release is off; grown by 2p + U).
 *                    Admission is always used + p + U <= cap; the over-
 *                    capacity count compares p + g with cap in every mode.
 *
 * Fidelity modes (Sec. 3.3 memory-aware scheduler and App. D):
 *   per_step = 1     between dispatch steps the loop runs step by step: on
 *                    each step a decoder whose running requests would pass
 *                    its capacity by taking one token each preempts its most
 *                    recently admitted request (never its last one), which
 *                    loses its tokens and goes to the head of the waiting
 *                    queue; each running request takes a token and those
 *                    reaching their true length complete; on every step
 *                    but a dispatch step the queue (preempted requests
 *                    first, the latest on top, then the order computed at
 *                    the last dispatch step) admits while used + p + U <=
 *                    cap, the first misfit blocking.
 *   beta >= 0        deferral: a request is dispatched at the first dispatch
 *                    step s at or after its arrival with arrival +
 *                    pred_delay <= s (its bound is available), by the
 *                    dispatch policy; one still without a bound beta steps
 *                    after arrival (or at the last dispatch step) goes round
 *                    robin (index mod D) with the horizon H as its bound
 *                    until its prediction arrives; at a dispatch step the
 *                    timed-out requests join their queues before the policy
 *                    dispatches the rest, in index order.  Every request in
 *                    the system whose prediction is not in yet is bounded
 *                    by H.
 *
 *   cfg                 host struct: N requests (1 .. INT32_MAX), D decoders
 *                       (1 .. 1024), horizon H steps, capacity cap tokens per
 *                       decoder, batch size, window size, alpha in parts per
 *                       million (0 < alpha_ppm < 10^6), max_wait steps,
 *                       and the three policy fields above.
 *   arrival_ms          [N] int64 arrival step.
 *   prompt, true_len, pred   [N] int32 prompt length (>= 0), true output
 *                       length (>= 1), predicted output length (>= 0).
 *   choice_out          [N] int32 decoder chosen for each request.
 *   q_out               [ceil(N / batch)] int32 quantile per batch (-1:
 *                       unbounded, round robin).
 *   stats_out           [ceil(N / batch)][4] int64 per batch: completions,
 *                       admissions, requests left waiting, decoders whose
 *                       running requests exceed capacity after advancing.
 *   pred_delay          [N] int32 steps from arrival until the request's
 *                       prediction (so its bound) is available, >= 0; read
 *                       only when cfg->beta >= 0 (then required).
 *   dec_stats_out       [D][4] int64 per decoder, or NULL: the waiting-queue
 *                       integral (requests waiting through each step from
 *                       the first dispatch step to the last, exclusive:
 *                       after batch b's admission times s_{b+1} - s_b when
 *                       admission happens at dispatch steps only), the
 *                       batches after whose advance its running requests
 *                       exceed capacity, its admissions, its preemptions.
 * The call runs the whole loop: it synchronises the stream once per batch
 * (to read the request counts that size the next launches) and at the end,
 * and returns the full status.  A negative length or decreasing arrival is
 * MAPS_E_RANGE before any batch runs.
 * ---------------------------------------------------------------------- */
typedef struct {
  int64_t N;
  int32_t D, H;
  int32_t cap;
  int32_t batch;
  int32_t window;
  uint32_t alpha_ppm;
  int32_t max_wait;
  int32_t dispatch_policy; /* MAPS_STREAM_MAPS / _MC / _RR / _LR */
  int32_t local_order;     /* MAPS_STREAM_SJF / _FCFS */
  int32_t accounting;      /* MAPS_STREAM_OCCUPANCY / _STAGED / _HELD */
  int32_t per_step;        /* 0: admission at dispatch steps; 1: every step, with preemption */
  int32_t beta;            /* < 0: bounds always available; >= 0: deferral timeout, steps */
} maps_stream_cfg;

#define MAPS_STREAM_MAPS 0
#define MAPS_STREAM_MC 1
#define MAPS_STREAM_RR 2
#define MAPS_STREAM_LR 3
#define MAPS_STREAM_SJF 0
#define MAPS_STREAM_FCFS 1
#define MAPS_STREAM_OCCUPANCY 0
#define MAPS_STREAM_STAGED 1
#define MAPS_STREAM_HELD 2

size_t maps_stream_workspace_size(const maps_stream_cfg *cfg);
int maps_stream_run(const maps_stream_cfg *cfg, const int64_t *arrival_ms,
                    const int32_t *prompt, const int32_t *true_len,
                    const int32_t *pred, const int32_t *pred_delay,
                    int32_t *choice_out, int32_t *q_out, int64_t *stats_out,
                    int64_t *dec_stats_out, void *ws, size_t ws_bytes,
                    void *stream);

/* ------------------------------------------------------------------------
 * Round-robin KV-pressure simulation and high-pressure interval metrics,
 * App. A (Eq. kv_demand, the routing equation, Eq. admission, Definition
 * of the high-pressure interval), for many workload realisations at once.
 *
 * Each realisation is n_req requests in arrival order.  Round robin sends
 * request i to decoder i mod N.  A request holds M = prompt + out_len KV
 * tokens while admitted; a decoder admits the head of its FIFO queue while
 * K + M(head) <= C.  Service is processor sharing at one token per t_tok,
 * taken at token granularity: a round gives each of the n admitted requests
 * one token and lasts n * t_tok; completions and then admissions happen at
 * round boundaries, and an idle decoder admits a request when it arrives.
 * A decoder is under high pressure while K * 1e6 >= theta_ppm * C.  Times
 * are integer microseconds.
 *
 *   cfg                 host struct (below).
 *   n_real              realisations (>= 1).
 *   arrival_us          [n_real][n_req] int64 arrival times, non-decreasing
 *                       within a realisation.
 *   prompt, out_len     [n_real][n_req] int32, prompt >= 0, out_len >= 1,
 *                       prompt + out_len <= C.
 *   admit_us, done_us   [n_real][n_req] int64 output: admission and
 *                       completion time of every request.
 *   stats               [n_real][N][6] int64 output per decoder: total time
 *                       under high pressure T_hp, longest high-pressure
 *                       interval B_hp, number of intervals C_hp, completed
 *                       requests, longest waiting queue at an arrival, total
 *                       waiting time (arrival to admission).
 *   t_sim               [n_real] int64 output: first arrival to last
 *                       completion (f_hp = T_hp / t_sim).
 * Inputs outside the domain, or more than 1,536 requests admitted at once on
 * one decoder, are MAPS_E_RANGE (via maps_check).
 * ---------------------------------------------------------------------- */
typedef struct {
  int64_t n_req;       /* requests per realisation */
  int32_t N;           /* decoders */
  int32_t C;           /* KV-token capacity per decoder */
  int32_t t_tok_us;    /* decode time per token, microseconds (>= 1) */
  uint32_t theta_ppm;  /* high-pressure threshold, parts per million of C (1 .. 1e6) */
} maps_rr_cfg;

size_t maps_rr_pressure_workspace_size(const maps_rr_cfg *cfg, int64_t n_real);
int maps_rr_pressure(const maps_rr_cfg *cfg, int64_t n_real, const int64_t *arrival_us,
                     const int32_t *prompt, const int32_t *out_len, int64_t *admit_us,
                     int64_t *done_us, int64_t *stats, int64_t *t_sim, void *ws,
                     size_t ws_bytes, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* MAPS_H */
