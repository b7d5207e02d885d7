/*
 * oracle_rr.c -- plain CPU reference of the round-robin KV-pressure
 * simulation of App. A and its high-pressure interval metrics.
 *
 * TEST INFRASTRUCTURE ONLY: used by the test suite and the benchmark's
 * CPU-baseline leg, never by the product path.  It shares no code with the
 * CUDA library.
 *
 * The model, step by step as App. A describes it:
 *   - requests arrive in order (arrival times given, microseconds) and round
 *     robin routes request i to decoder i mod N (App. A, routing equation);
 *   - request r holds M(r) = L_p + L_out KV tokens while admitted
 *     (Eq. kv_demand);
 *   - a decoder admits the head of its FIFO waiting queue while
 *     K_d + M(head) <= C (Eq. admission), K_d being the tokens its admitted
 *     requests hold;
 *   - service is processor sharing: a decoder produces one token every
 *     t_tok, shared evenly by its admitted requests.
 * Readings where App. A leaves the detail open (the same on the GPU side):
 *   - processor sharing is taken at token granularity: with n requests
 *     admitted, a round gives each of them one token and lasts n * t_tok, so
 *     every time stays an exact integer; a request completes at the end of
 *     its L_out-th round;
 *   - completions and admissions happen at round boundaries, completions
 *     first; an idle decoder admits a request when it arrives;
 *   - K_d(t) is right-continuous: the value after every change at t.  The
 *     decoder is in the high-pressure state when K_d * 1e6 >= theta_ppm * C
 *     (Definition of the HP interval, theta in parts per million);
 *   - a request whose footprint exceeds C could never be admitted: the call
 *     rejects such input (range error).
 * Outputs per request: admission and completion times.  Per decoder: T_hp
 * (total time in the high-pressure state), B_hp (longest HP interval), C_hp
 * (number of HP intervals), completed requests, the longest waiting queue
 * seen at an arrival, and the total waiting time (arrival to admission).
 * T_sim runs from the first arrival to the last completion.
 *
 * This is the literal form: the simulation advances round by round and
 * every admitted request gains one token per round.  No event skipping.
 */
#include "oracle.h"

#include <stdlib.h>

static void hp_update(int64_t K, int64_t C, uint32_t theta_ppm, int64_t t,
                      int *in_hp, int64_t *t_s, int64_t *st)
{
    int now = K * 1000000 >= (int64_t)theta_ppm * C;
    if (now && !*in_hp) {
        *in_hp = 1;
        *t_s = t;
    } else if (!now && *in_hp) {
        int64_t len = t - *t_s;
        *in_hp = 0;
        st[0] += len;             /* T_hp */
        if (len > st[1]) st[1] = len; /* B_hp */
        st[2] += 1;               /* C_hp */
    }
}

int oracle_rr_pressure(const oracle_rr_cfg *cfg, const int64_t *arrival_us,
                       const int32_t *prompt, const int32_t *out_len,
                       int64_t *admit_us, int64_t *done_us, int64_t *stats,
                       int64_t *t_sim)
{
    if (cfg == NULL || cfg->n_req < 1 || cfg->N < 1 || cfg->C < 1 ||
        cfg->t_tok_us < 1 || cfg->theta_ppm == 0 || cfg->theta_ppm > 1000000u ||
        arrival_us == NULL || prompt == NULL || out_len == NULL ||
        admit_us == NULL || done_us == NULL || stats == NULL || t_sim == NULL)
        return ORACLE_E_INVALID;
    const int64_t n = cfg->n_req, C = cfg->C, tok = cfg->t_tok_us;
    const int32_t N = cfg->N;
    for (int64_t i = 0; i < n; ++i)
        if (prompt[i] < 0 || out_len[i] < 1 || arrival_us[i] < 0 ||
            (int64_t)prompt[i] + out_len[i] > C ||
            (i > 0 && arrival_us[i] < arrival_us[i - 1]))
            return ORACLE_E_RANGE;

    int64_t *rem = (int64_t *)malloc((size_t)n * sizeof(int64_t));
    int64_t *run = (int64_t *)malloc((size_t)n * sizeof(int64_t));
    if (rem == NULL || run == NULL) {
        free(rem);
        free(run);
        return ORACLE_E_INVALID;
    }
    int64_t last_done = 0;
    for (int32_t d = 0; d < N; ++d) {
        int64_t *st = stats + (int64_t)d * 6;
        for (int q = 0; q < 6; ++q)
            st[q] = 0;
        if (d >= n)
            continue;
        /* decoder d's requests: i = d, d + N, d + 2N, ... in arrival order */
        int64_t head = d;          /* first request not yet admitted */
        int64_t n_run = 0, K = 0;  /* admitted, their tokens */
        int64_t t = arrival_us[d];
        int in_hp = 0;
        int64_t t_s = 0;
        for (;;) {
            /* admissions at t: the FIFO head, while it has arrived and fits */
            while (head < n && arrival_us[head] <= t &&
                   K + prompt[head] + out_len[head] <= C) {
                admit_us[head] = t;
                rem[head] = out_len[head];
                run[n_run++] = head;
                K += (int64_t)prompt[head] + out_len[head];
                head += N;
            }
            hp_update(K, C, cfg->theta_ppm, t, &in_hp, &t_s, st);
            if (n_run == 0) {
                if (head >= n)
                    break;
                t = arrival_us[head]; /* idle until the head arrives */
                continue;
            }
            /* one round: every admitted request gains a token */
            t += n_run * tok;
            int64_t w = 0;
            for (int64_t j = 0; j < n_run; ++j) {
                int64_t i = run[j];
                if (--rem[i] == 0) {
                    done_us[i] = t;
                    K -= (int64_t)prompt[i] + out_len[i];
                    st[3] += 1;
                    if (t > last_done)
                        last_done = t;
                } else {
                    run[w++] = i;
                }
            }
            n_run = w;
        }
        /* waiting: total, and the longest queue seen at an arrival (the
         * requests arrived by then and not yet admitted) */
        for (int64_t i = d; i < n; i += N) {
            st[5] += admit_us[i] - arrival_us[i];
            int64_t queued = 0;
            for (int64_t j = d; j <= i; j += N)
                if (admit_us[j] > arrival_us[i])
                    queued += 1;
            if (queued > st[4])
                st[4] = queued;
        }
    }
    *t_sim = last_done - arrival_us[0];
    free(rem);
    free(run);
    return ORACLE_OK;
}
