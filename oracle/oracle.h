/*
 * oracle.h -- plain CPU reference of the MAPS scheduler hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may include, link,
 * load or execute this code; only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg use it.  It shares no code, header, table or
 * helper with the CUDA library: the two meet only through the seeded input
 * generator, which holds none of the scheduler's arithmetic.
 *
 * Every routine computes the quantity by its definition, in 64-bit integer
 * arithmetic, one element at a time, in the order the paper states it.  All
 * pointers are host pointers owned by the caller.
 *
 * Status codes mirror the product library so results can be compared
 * one-to-one:  0 ok, -1 invalid argument, -2 value outside the int32 range
 * or the input domain, -3 conformal quantile unbounded (rank > n).
 */
#ifndef MAPS_ORACLE_H
#define MAPS_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORACLE_OK 0
#define ORACLE_E_INVALID (-1)
#define ORACLE_E_RANGE (-2)
#define ORACLE_E_UNBOUNDED (-3)

#define ORACLE_MODE_SNAPSHOT 0
#define ORACLE_MODE_SEQUENTIAL 1
#define ORACLE_MODE_ALG1_SNAPSHOT 2
#define ORACLE_MODE_ALG1_SEQUENTIAL 3

/* Sec. 3.2: the conformal rank ceil((1-alpha)(n+1)), alpha = alpha_ppm/1e6. */
int64_t oracle_rank(int64_t n, uint32_t alpha_ppm);

/* Sec. 3.2, Eq. (nonconformity) and the quantile that follows it:
 * s_i = max(0, L_i - Lhat_i); q = the rank-th smallest s. */
int oracle_calibrate(const int32_t *true_len, const int32_t *pred_len,
                     int64_t n, uint32_t alpha_ppm, int64_t *q_out);

/* Eq. (conformal_upper): U = Lhat + q for every query prediction. */
int oracle_bound(const int32_t *pred, int64_t m, int64_t q, int32_t *bound_out);

/* Projected KV-token occupancy over the step horizon:
 * K_k(t) = sum over residents r of decoder k with t < e_r of (b_r + t),
 * b_r = p_r + g_r + 1, e_r = min(max(U_r - g_r, 1), H).  K is [D][H]. */
int oracle_occupancy(int32_t D, int32_t H, const int64_t *res_off, int64_t R,
                     const int32_t *prompt, const int32_t *gen,
                     const int32_t *bound, int32_t *K_out);

/* One occupancy cell by the sum definition (for sampled checks at scale). */
int64_t oracle_occupancy_cell(int32_t H, const int64_t *res_off, int32_t k,
                              int32_t t, const int32_t *prompt,
                              const int32_t *gen, const int32_t *bound);

/* Sec. 3.3 memory-aware dispatch and Algorithm 1 (all four modes). */
int oracle_dispatch(int32_t mode, int32_t D, int32_t H, int32_t S,
                    int32_t *K, const int32_t *cap, int32_t *Q,
                    const int64_t *res_off, int64_t R, const int32_t *prompt,
                    const int32_t *gen, const int32_t *bound, int64_t J,
                    const int32_t *cand_prompt, const int32_t *cand_bound,
                    int32_t *choice_out, int64_t *headroom_out);

/* Sec. 3.3 local SJF order with max-wait promotion. */
int oracle_order_local(int64_t N, int32_t D, const int32_t *dec,
                       const int32_t *bound, const int32_t *wait,
                       const int32_t *arrival, int32_t max_wait,
                       int32_t *perm_out, int64_t *seg_off_out);

/* The streaming loop: batches of arrivals dispatched sequentially with
 * per-batch recalibration over a sliding window of completions. */
typedef struct {
    int64_t N;          /* requests */
    int32_t D, H;       /* decoders, horizon (steps) */
    int32_t cap;        /* KV-token capacity per decoder */
    int32_t batch;      /* requests per dispatch batch */
    int32_t window;     /* calibration window (completed requests) */
    uint32_t alpha_ppm; /* miscoverage * 1e6 */
    int32_t max_wait;   /* promotion threshold, steps */
    int32_t dispatch;   /* 0 MAPS (min Q among feasible, else most headroom),
                           1 MC (most headroom), 2 round robin, 3 least requests */
    int32_t local;      /* 0 SJF with max-wait promotion, 1 FCFS */
    int32_t accounting; /* admission counts running requests at 0 their tokens,
                           1 prompt + reserved output (staged release),
                           2 reserved prompt + prompt + reserved output */
    int32_t per_step;   /* 0 admission at dispatch steps only; 1 every step,
                           with preemption of the latest admitted request */
    int32_t beta;       /* timeout (steps) for a bound not yet available;
                           < 0: every bound is available at dispatch */
} oracle_stream_cfg;

/* pred_delay[N] (may be NULL: 0): steps from arrival until the request's
 * prediction, and so its bound, is available (used when beta >= 0).
 * Outputs: choice[N]; per batch b: q[b] (-1 if unbounded -> round robin),
 * stats[4b..4b+3] = completed, admitted, waiting after admission,
 * decoders over capacity after advancing; per decoder k (dec_stats may be
 * NULL): dec_stats[4k..4k+3] = waiting requests x steps summed over the
 * batches (the time-weighted queue length times the span), batches in which
 * it was over capacity after advancing, admissions, preemptions. */
int oracle_stream(const oracle_stream_cfg *cfg, const int64_t *arrival_ms,
                  const int32_t *prompt, const int32_t *true_len,
                  const int32_t *pred, const int32_t *pred_delay,
                  int32_t *choice_out, int32_t *q_out,
                  int64_t *stats_out, int64_t *dec_stats_out);

/* Round-robin KV-pressure simulation of App. A (oracle_rr.c). */
typedef struct {
    int64_t n_req;       /* requests, in arrival order */
    int32_t N;           /* decoders (round robin over them) */
    int32_t C;           /* KV-token capacity per decoder */
    int32_t t_tok_us;    /* decode time per token, microseconds */
    uint32_t theta_ppm;  /* high-pressure threshold * 1e6 */
} oracle_rr_cfg;

/* Outputs: admit_us[n_req], done_us[n_req]; stats[6d .. 6d+5] = T_hp,
 * B_hp, C_hp, completed, longest queue, total wait of decoder d; *t_sim. */
int oracle_rr_pressure(const oracle_rr_cfg *cfg, const int64_t *arrival_us,
                       const int32_t *prompt, const int32_t *out_len,
                       int64_t *admit_us, int64_t *done_us, int64_t *stats,
                       int64_t *t_sim);

#ifdef __cplusplus
}
#endif
#endif
