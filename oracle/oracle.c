/*
 * oracle.c -- plain CPU reference of the MAPS scheduler hot path.
 *
 * TEST INFRASTRUCTURE ONLY: used by the test suite, the smoke check and the
 * benchmark's CPU-baseline leg, never by the product path.  It shares no
 * code with the CUDA library.
 *
 * Each routine is the definition written out, in 64-bit integer arithmetic:
 *   - the conformal quantile sorts all scores and reads the rank-th one;
 *   - the occupancy adds every resident's footprint to every step it covers;
 *   - each (candidate, decoder) score takes the maximum over the steps the
 *     candidate is live, step by step;
 *   - the local order sorts with the full comparator.
 * No blocking, fusion or reordering beyond that.  Library primitives used as
 * steps: qsort (a comparison sort) and memset.
 *
 * Readings of the paper taken here (where it is silent):
 *   - step convention: at step t in [0, H) a resident with p prompt tokens and
 *     g generated tokens holds p + g + t + 1 KV slots and is live while
 *     t < U - g; one already past its bound stays live for one step; a
 *     candidate holds p + t + 1 while t < U (at least one step); everything is
 *     truncated at the horizon H;
 *   - dispatch rule in horizon form: feasible iff the candidate's peak
 *     projected occupancy fits the capacity; feasible decoders are ranked by
 *     queue length, infeasible ones by headroom; ties go to the lowest index;
 *   - alpha crosses the interface in parts per million so the rank
 *     ceil((1-alpha)(n+1)) is exact.
 */
#include "oracle.h"

#include <stdlib.h>
#include <string.h>

#define I32_MAX 2147483647LL
#define KEY_INFEASIBLE_BASE ((int64_t)1 << 62)

/* ---------------------------------------------------------------------- */
/* Sec. 3.2 -- uncertainty-aware calibration                               */
/* ---------------------------------------------------------------------- */

int64_t oracle_rank(int64_t n, uint32_t alpha_ppm)
{
    /* ceil((1 - a/1e6) * (n + 1)) written as an exact integer ceiling. */
    int64_t num = (int64_t)(1000000u - alpha_ppm) * (n + 1);
    return (num + 999999) / 1000000;
}

static int cmp_i64(const void *a, const void *b)
{
    int64_t x = *(const int64_t *)a, y = *(const int64_t *)b;
    return (x > y) - (x < y);
}

int oracle_calibrate(const int32_t *true_len, const int32_t *pred_len,
                     int64_t n, uint32_t alpha_ppm, int64_t *q_out)
{
    if (q_out == NULL || n < 0 || n > ((int64_t)1 << 40) || alpha_ppm == 0 ||
        alpha_ppm >= 1000000u || (n > 0 && (true_len == NULL || pred_len == NULL)))
        return ORACLE_E_INVALID;
    int64_t k = oracle_rank(n, alpha_ppm);
    if (k > n)
        return ORACLE_E_UNBOUNDED; /* the quantile is +infinity */
    int64_t *s = (int64_t *)malloc((size_t)n * sizeof(int64_t));
    if (s == NULL)
        return ORACLE_E_INVALID;
    for (int64_t i = 0; i < n; ++i) {
        /* Eq. (nonconformity): one-sided score, positive only on
         * underestimation. */
        int64_t d = (int64_t)true_len[i] - (int64_t)pred_len[i];
        s[i] = d > 0 ? d : 0;
    }
    qsort(s, (size_t)n, sizeof(int64_t), cmp_i64);
    int64_t q = s[k - 1]; /* k-th smallest, 1-indexed */
    free(s);
    if (q > I32_MAX)
        return ORACLE_E_RANGE;
    *q_out = q;
    return ORACLE_OK;
}

int oracle_bound(const int32_t *pred, int64_t m, int64_t q, int32_t *bound_out)
{
    if (m < 0 || q < 0 || q > I32_MAX || (m > 0 && (pred == NULL || bound_out == NULL)))
        return ORACLE_E_INVALID;
    int status = ORACLE_OK;
    for (int64_t i = 0; i < m; ++i) {
        int64_t u = (int64_t)pred[i] + q; /* Eq. (conformal_upper) */
        if (u > I32_MAX) {
            status = ORACLE_E_RANGE;
            u = I32_MAX;
        }
        bound_out[i] = (int32_t)u;
    }
    return status;
}

/* ---------------------------------------------------------------------- */
/* Projected KV-token occupancy over the step horizon                      */
/* (footprint M(r) = L_p + L_out of Eq. (kv_demand), occupancy K_d(t) of   */
/*  Eq. (admission), extended over steps t = 0 .. H-1)                     */
/* ---------------------------------------------------------------------- */

/* Residents of decoder k are [res_off[k], res_off[k+1]); the offsets must be
 * non-decreasing inside [0, R]. */
static int offsets_ok(int32_t D, const int64_t *res_off, int64_t R)
{
    if (res_off[0] < 0 || res_off[D] > R)
        return 0;
    for (int32_t k = 0; k < D; ++k)
        if (res_off[k + 1] < res_off[k])
            return 0;
    return 1;
}

/* End step (exclusive) and t=0 footprint of one resident; returns 0 if the
 * resident is outside the domain (negative length). */
static int resident_terms(int32_t H, int32_t p, int32_t g, int32_t U,
                          int64_t *b, int64_t *e)
{
    if (p < 0 || g < 0 || U < 0)
        return 0;
    *b = (int64_t)p + (int64_t)g + 1;
    int64_t end = (int64_t)U - (int64_t)g;
    if (end < 1)
        end = 1;
    if (end > H)
        end = H;
    *e = end;
    return 1;
}

int oracle_occupancy(int32_t D, int32_t H, const int64_t *res_off, int64_t R,
                     const int32_t *prompt, const int32_t *gen,
                     const int32_t *bound, int32_t *K_out)
{
    if (D < 1 || H < 1 || R < 0 || res_off == NULL || K_out == NULL ||
        (R > 0 && (prompt == NULL || gen == NULL || bound == NULL)))
        return ORACLE_E_INVALID;
    if (!offsets_ok(D, res_off, R))
        return ORACLE_E_RANGE;
    int status = ORACLE_OK;
    int64_t *acc = (int64_t *)malloc((size_t)H * sizeof(int64_t));
    if (acc == NULL)
        return ORACLE_E_INVALID;
    for (int32_t k = 0; k < D; ++k) {
        memset(acc, 0, (size_t)H * sizeof(int64_t));
        for (int64_t r = res_off[k]; r < res_off[k + 1]; ++r) {
            int64_t b, e;
            if (!resident_terms(H, prompt[r], gen[r], bound[r], &b, &e)) {
                status = ORACLE_E_RANGE;
                continue;
            }
            for (int64_t t = 0; t < e; ++t)
                acc[t] += b + t;
        }
        for (int32_t t = 0; t < H; ++t) {
            int64_t v = acc[t];
            if (v > I32_MAX) {
                status = ORACLE_E_RANGE;
                v = I32_MAX;
            }
            K_out[(int64_t)k * H + t] = (int32_t)v;
        }
    }
    free(acc);
    return status;
}

int64_t oracle_occupancy_cell(int32_t H, const int64_t *res_off, int32_t k,
                              int32_t t, const int32_t *prompt,
                              const int32_t *gen, const int32_t *bound)
{
    int64_t sum = 0;
    for (int64_t r = res_off[k]; r < res_off[k + 1]; ++r) {
        int64_t b, e;
        if (!resident_terms(H, prompt[r], gen[r], bound[r], &b, &e))
            return -1;
        if (t < e)
            sum += b + t;
    }
    return sum;
}

/* ---------------------------------------------------------------------- */
/* Sec. 3.3 memory-aware dispatch, Algorithm 1                             */
/* ---------------------------------------------------------------------- */

static int64_t ceil_div(int64_t a, int64_t s) { return (a + s - 1) / s; }

/* Horizon form of the feasibility test: the candidate's KV footprint ramp
 * p + t + 1 (t < u) on top of the decoder's projected occupancy K(t). */
static int64_t candidate_peak(const int32_t *Krow, int64_t p, int64_t u)
{
    int64_t m = INT64_MIN;
    for (int64_t t = 0; t < u; ++t) {
        int64_t v = (int64_t)Krow[t] + p + t + 1;
        if (v > m)
            m = v;
    }
    return m;
}

static int dispatch_horizon(int sequential, int mc, int32_t D, int32_t H, int32_t *K,
                            const int32_t *cap, int32_t *Q, int64_t J,
                            const int32_t *cand_prompt,
                            const int32_t *cand_bound, int32_t *choice_out,
                            int64_t *headroom_out)
{
    int status = ORACLE_OK;
    for (int64_t i = 0; i < (int64_t)D * H; ++i)
        if (K[i] < 0)
            return ORACLE_E_RANGE;
    for (int64_t j = 0; j < J; ++j) {
        int64_t p = cand_prompt[j], U = cand_bound[j];
        if (p < 0 || U < 0) {
            status = ORACLE_E_RANGE;
            choice_out[j] = -1;
            if (headroom_out)
                headroom_out[j] = 0;
            continue;
        }
        int64_t u = U < 1 ? 1 : (U > H ? H : U);
        int32_t best = -1;
        int64_t best_key = 0, best_h = 0;
        for (int32_t k = 0; k < D; ++k) {
            int64_t peak = candidate_peak(K + (int64_t)k * H, p, u);
            int64_t h = (int64_t)cap[k] - peak;
            /* Feasible decoders compete on queue length (min Q); only when
             * none is feasible does the most headroom win.  The MC variant
             * (Sec. 4 ablation MQ->MC) ranks every decoder by headroom. */
            int64_t key = h >= 0 && !mc ? (int64_t)Q[k] : KEY_INFEASIBLE_BASE - h;
            if (best < 0 || key < best_key) {
                best = k;
                best_key = key;
                best_h = h;
            }
        }
        choice_out[j] = best;
        if (headroom_out)
            headroom_out[j] = best_h;
        if (sequential) {
            /* Reserve the footprint at the chosen decoder before the next
             * candidate is scored. */
            int32_t *row = K + (int64_t)best * H;
            for (int64_t t = 0; t < u; ++t) {
                int64_t v = (int64_t)row[t] + p + t + 1;
                if (v > I32_MAX) {
                    status = ORACLE_E_RANGE;
                    v = I32_MAX;
                }
                row[t] = (int32_t)v;
            }
            if (Q[best] == (int32_t)I32_MAX)
                status = ORACLE_E_RANGE;
            else
                Q[best] += 1;
        }
    }
    return status;
}

static int dispatch_alg1(int sequential, int32_t D, int32_t S,
                         const int32_t *cap, int32_t *Q,
                         const int64_t *res_off, const int32_t *prompt,
                         const int32_t *gen, const int32_t *bound, int64_t J,
                         const int32_t *cand_prompt, const int32_t *cand_bound,
                         int32_t *choice_out, int64_t *headroom_out)
{
    int status = ORACLE_OK;
    int64_t *B_eff = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    if (B_eff == NULL)
        return ORACLE_E_INVALID;
    for (int32_t k = 0; k < D; ++k) {
        /* B_eff = B_free - B_res: the capacity in blocks minus what every
         * ongoing request holds or has reserved at its bound. */
        int64_t held = 0;
        for (int64_t r = res_off[k]; r < res_off[k + 1]; ++r) {
            int64_t p = prompt[r], g = gen[r], U = bound[r];
            if (p < 0 || g < 0 || U < 0) {
                status = ORACLE_E_RANGE;
                continue;
            }
            int64_t tokens = p + (U > g + 1 ? U : g + 1);
            held += ceil_div(tokens, S);
        }
        B_eff[k] = (int64_t)cap[k] / S - held;
    }
    for (int64_t j = 0; j < J; ++j) {
        int64_t p = cand_prompt[j], U = cand_bound[j];
        if (p < 0 || U < 0) {
            status = ORACLE_E_RANGE;
            choice_out[j] = -1;
            if (headroom_out)
                headroom_out[j] = 0;
            continue;
        }
        int64_t need = ceil_div(p + U, S); /* Eq. (feasibility) */
        int32_t best = -1;
        int64_t best_key = 0;
        for (int32_t k = 0; k < D; ++k) {
            int64_t h = B_eff[k] - need;
            /* Alg. 1: argmin Q over the feasible set, else argmax B_eff. */
            int64_t key = h >= 0 ? (int64_t)Q[k] : KEY_INFEASIBLE_BASE - h;
            if (best < 0 || key < best_key) {
                best = k;
                best_key = key;
            }
        }
        choice_out[j] = best;
        if (headroom_out)
            headroom_out[j] = B_eff[best] - need;
        if (sequential) {
            B_eff[best] -= need;
            if (Q[best] == (int32_t)I32_MAX)
                status = ORACLE_E_RANGE;
            else
                Q[best] += 1;
        }
    }
    free(B_eff);
    return status;
}

int oracle_dispatch(int32_t mode, int32_t D, int32_t H, int32_t S,
                    int32_t *K, const int32_t *cap, int32_t *Q,
                    const int64_t *res_off, int64_t R, const int32_t *prompt,
                    const int32_t *gen, const int32_t *bound, int64_t J,
                    const int32_t *cand_prompt, const int32_t *cand_bound,
                    int32_t *choice_out, int64_t *headroom_out)
{
    if (D < 1 || J < 0 || cap == NULL || Q == NULL ||
        (J > 0 && (cand_prompt == NULL || cand_bound == NULL || choice_out == NULL)))
        return ORACLE_E_INVALID;
    for (int32_t k = 0; k < D; ++k)
        if (cap[k] < 0 || Q[k] < 0)
            return ORACLE_E_RANGE;
    if (mode == ORACLE_MODE_SNAPSHOT || mode == ORACLE_MODE_SEQUENTIAL) {
        if (H < 1 || K == NULL)
            return ORACLE_E_INVALID;
        return dispatch_horizon(mode == ORACLE_MODE_SEQUENTIAL, 0, D, H, K, cap, Q,
                                J, cand_prompt, cand_bound, choice_out,
                                headroom_out);
    }
    if (mode == ORACLE_MODE_ALG1_SNAPSHOT || mode == ORACLE_MODE_ALG1_SEQUENTIAL) {
        if (S < 1 || res_off == NULL || R < 0 ||
            (R > 0 && (prompt == NULL || gen == NULL || bound == NULL)))
            return ORACLE_E_INVALID;
        if (!offsets_ok(D, res_off, R))
            return ORACLE_E_RANGE;
        return dispatch_alg1(mode == ORACLE_MODE_ALG1_SEQUENTIAL, D, S, cap, Q,
                             res_off, prompt, gen, bound, J, cand_prompt,
                             cand_bound, choice_out, headroom_out);
    }
    return ORACLE_E_INVALID;
}

/* ---------------------------------------------------------------------- */
/* Sec. 3.3 local SJF reordering with the maximum-waiting-time promotion   */
/* ---------------------------------------------------------------------- */

typedef struct {
    int64_t dec, not_promoted, primary, arrival, idx;
} order_item;

static int cmp_order(const void *a, const void *b)
{
    const order_item *x = (const order_item *)a, *y = (const order_item *)b;
    if (x->dec != y->dec)
        return x->dec < y->dec ? -1 : 1;
    if (x->not_promoted != y->not_promoted)
        return x->not_promoted < y->not_promoted ? -1 : 1;
    if (x->primary != y->primary)
        return x->primary < y->primary ? -1 : 1;
    if (x->arrival != y->arrival)
        return x->arrival < y->arrival ? -1 : 1;
    return (x->idx > y->idx) - (x->idx < y->idx);
}

int oracle_order_local(int64_t N, int32_t D, const int32_t *dec,
                       const int32_t *bound, const int32_t *wait,
                       const int32_t *arrival, int32_t max_wait,
                       int32_t *perm_out, int64_t *seg_off_out)
{
    if (N < 0 || N > I32_MAX || D < 1 || seg_off_out == NULL ||
        (N > 0 && (dec == NULL || bound == NULL || wait == NULL ||
                   arrival == NULL || perm_out == NULL)))
        return ORACLE_E_INVALID;
    order_item *it = (order_item *)malloc((size_t)(N > 0 ? N : 1) * sizeof(order_item));
    if (it == NULL)
        return ORACLE_E_INVALID;
    int status = ORACLE_OK;
    for (int64_t i = 0; i < N; ++i) {
        if (dec[i] < 0 || dec[i] >= D || bound[i] < 0 || arrival[i] < 0)
            status = ORACLE_E_RANGE;
        /* Requests waiting longer than the threshold are promoted ahead of
         * the SJF order and served first-come-first-served among
         * themselves; the rest follow argsort of the bound, ties by
         * arrival. */
        int promoted = wait[i] > max_wait;
        it[i].dec = dec[i];
        it[i].not_promoted = !promoted;
        it[i].primary = promoted ? arrival[i] : bound[i];
        it[i].arrival = arrival[i];
        it[i].idx = i;
    }
    if (status != ORACLE_OK) {
        free(it);
        return status;
    }
    qsort(it, (size_t)N, sizeof(order_item), cmp_order);
    for (int32_t k = 0; k <= D; ++k)
        seg_off_out[k] = 0;
    for (int64_t i = 0; i < N; ++i) {
        perm_out[i] = (int32_t)it[i].idx;
        seg_off_out[it[i].dec + 1] += 1;
    }
    for (int32_t k = 0; k < D; ++k)
        seg_off_out[k + 1] += seg_off_out[k];
    free(it);
    return ORACLE_OK;
}

/* ---------------------------------------------------------------------- */
/* The streaming loop                                                      */
/* ---------------------------------------------------------------------- */

enum { ST_PENDING = 0, ST_WAITING = 1, ST_RUNNING = 2, ST_DONE = 3 };

typedef struct {
    int64_t step, id;
} completion;

static int cmp_completion(const void *a, const void *b)
{
    const completion *x = (const completion *)a, *y = (const completion *)b;
    if (x->step != y->step)
        return x->step < y->step ? -1 : 1;
    return (x->id > y->id) - (x->id < y->id);
}

/* Per-step mode: each decoder's running requests in admission order (a
 * doubly linked list; the tail is the most recently admitted), the requests
 * preempted since the last dispatch step (a stack: the latest on top, the
 * head of the waiting queue), and the waiting queue as ordered at the last
 * dispatch step (positions [qhead, qend) of that order). */
typedef struct {
    int64_t *next, *prev;   /* [N] running-list links, -1 at the ends */
    int64_t *head, *tail;   /* [D] */
    int64_t *pnext;         /* [N] preempted-stack links */
    int64_t *ptop;          /* [D] */
    int64_t *qhead, *qend;  /* [D] */
} step_lists;

static void run_append(step_lists *L, int32_t k, int64_t id)
{
    L->next[id] = -1;
    L->prev[id] = L->tail[k];
    if (L->tail[k] >= 0)
        L->next[L->tail[k]] = id;
    else
        L->head[k] = id;
    L->tail[k] = id;
}

static void run_unlink(step_lists *L, int32_t k, int64_t id)
{
    if (L->prev[id] >= 0)
        L->next[L->prev[id]] = L->next[id];
    else
        L->head[k] = L->next[id];
    if (L->next[id] >= 0)
        L->prev[L->next[id]] = L->prev[id];
    else
        L->tail[k] = L->prev[id];
}

/* What admission counts a running request for (cfg->accounting). */
static int64_t held_tokens(int32_t accounting, int64_t p, int64_t g, int64_t r)
{
    int64_t out_part = r > g ? r : g;
    return accounting == 0 ? p + g : accounting == 1 ? p + out_part : 2 * p + out_part;
}

/* What an admission adds to that count. */
static int64_t admit_tokens(int32_t accounting, int64_t p, int64_t u)
{
    return accounting == 0 ? p : accounting == 1 ? p + u : 2 * p + u;
}

int oracle_stream(const oracle_stream_cfg *cfg, const int64_t *arrival_ms,
                  const int32_t *prompt, const int32_t *true_len,
                  const int32_t *pred, const int32_t *pred_delay,
                  int32_t *choice_out, int32_t *q_out,
                  int64_t *stats_out, int64_t *dec_stats_out)
{
    if (cfg == NULL || cfg->N < 1 || cfg->N > I32_MAX || cfg->D < 1 ||
        cfg->H < 1 || cfg->cap < 0 || cfg->batch < 1 || cfg->window < 1 ||
        cfg->alpha_ppm == 0 || cfg->alpha_ppm >= 1000000u ||
        cfg->dispatch < 0 || cfg->dispatch > 3 || cfg->local < 0 || cfg->local > 1 ||
        cfg->accounting < 0 || cfg->accounting > 2 || cfg->per_step < 0 ||
        cfg->per_step > 1)
        return ORACLE_E_INVALID;
    const int64_t N = cfg->N;
    const int32_t D = cfg->D, H = cfg->H, Bsz = cfg->batch, Wn = cfg->window;
    const int64_t nb = (N + Bsz - 1) / Bsz;
    /* deferral: a bound becomes available pred_delay steps after arrival */
    const int defer = cfg->beta >= 0 && pred_delay != NULL;
    for (int64_t i = 0; i < N; ++i)
        if (prompt[i] < 0 || true_len[i] < 1 || pred[i] < 0 ||
            (pred_delay != NULL && pred_delay[i] < 0) ||
            (i > 0 && arrival_ms[i] < arrival_ms[i - 1]))
            return ORACLE_E_RANGE;

    int status = ORACLE_OK;
    int8_t *st = (int8_t *)calloc((size_t)N, 1);
    int32_t *g = (int32_t *)calloc((size_t)N, sizeof(int32_t));
    int32_t *dec = (int32_t *)calloc((size_t)N, sizeof(int32_t));
    int32_t *U = (int32_t *)calloc((size_t)N, sizeof(int32_t));
    int64_t *disp = (int64_t *)calloc((size_t)N, sizeof(int64_t));
    int64_t *act = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    completion *done = (completion *)malloc((size_t)N * sizeof(completion));
    int32_t *win_true = (int32_t *)malloc((size_t)Wn * sizeof(int32_t));
    int32_t *win_pred = (int32_t *)malloc((size_t)Wn * sizeof(int32_t));
    int32_t *K = (int32_t *)malloc((size_t)D * H * sizeof(int32_t));
    int32_t *capv = (int32_t *)malloc((size_t)D * sizeof(int32_t));
    int32_t *Q = (int32_t *)malloc((size_t)D * sizeof(int32_t));
    int64_t *off = (int64_t *)malloc((size_t)(D + 1) * sizeof(int64_t));
    int64_t *used = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    int64_t *seg = (int64_t *)malloc((size_t)(D + 1) * sizeof(int64_t));
    /* per-batch resident / waiting scratch, sized for the worst case */
    int32_t *rp = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *rg = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *rU = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int64_t *wid = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    int32_t *wdec = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *wU = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *wwait = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *warr = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *wperm = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int64_t *cid = (int64_t *)malloc((size_t)N * sizeof(int64_t));  /* dispatched by the policy */
    int32_t *cp = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *cU = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int32_t *cch = (int32_t *)malloc((size_t)N * sizeof(int32_t));
    int64_t *hr = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    int64_t *pend = (int64_t *)malloc((size_t)N * sizeof(int64_t)); /* arrived, not dispatched */
    int32_t *res_u = (int32_t *)calloc((size_t)N, sizeof(int32_t)); /* bound reserved at admission */
    int64_t *occ = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    int64_t *nreq = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    int64_t *dst = (int64_t *)calloc((size_t)D * 4, sizeof(int64_t));
    step_lists L;
    L.next = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    L.prev = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    L.pnext = (int64_t *)malloc((size_t)N * sizeof(int64_t));
    L.head = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    L.tail = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    L.ptop = (int64_t *)malloc((size_t)D * sizeof(int64_t));
    L.qhead = (int64_t *)calloc((size_t)D, sizeof(int64_t));
    L.qend = (int64_t *)calloc((size_t)D, sizeof(int64_t));
    if (!st || !g || !dec || !U || !disp || !act || !done || !win_true ||
        !win_pred || !K || !capv || !Q || !off || !used || !seg || !rp || !rg ||
        !rU || !wid || !wdec || !wU || !wwait || !warr || !wperm || !cid || !cp ||
        !cU || !cch || !hr || !pend || !res_u || !occ || !nreq || !dst ||
        !L.next || !L.prev || !L.pnext || !L.head || !L.tail || !L.ptop ||
        !L.qhead || !L.qend) {
        status = ORACLE_E_INVALID;
        goto out;
    }
    for (int32_t k = 0; k < D; ++k) {
        capv[k] = cfg->cap;
        L.head[k] = L.tail[k] = L.ptop[k] = -1;
    }

    int64_t nact = 0, npend = 0, win_len = 0, win_head = 0;
    int64_t prev_s = arrival_ms[(N < Bsz ? N : Bsz) - 1];
    for (int64_t b = 0; b < nb; ++b) {
        const int64_t lo = b * Bsz, hi = (lo + Bsz < N) ? lo + Bsz : N;
        const int64_t s = arrival_ms[hi - 1]; /* dispatch step of batch b */
        const int64_t delta = s - prev_s;
        int64_t ndone = 0, admitted = 0;

        /* 1. Advance every running request by delta decode steps (one token
         *    per step); a request finishes when it reaches its true length. */
        if (!cfg->per_step) {
            for (int64_t a = 0; a < nact; ++a) {
                int64_t id = act[a];
                if (st[id] != ST_RUNNING)
                    continue;
                int64_t rem = (int64_t)true_len[id] - g[id];
                if (rem <= delta) {
                    st[id] = ST_DONE;
                    done[ndone].step = prev_s + rem;
                    done[ndone].id = id;
                    ++ndone;
                } else {
                    g[id] += (int32_t)delta;
                }
            }
        } else {
            /* Per-step mode: steps prev_s + 1 .. s one at a time, each
             * decoder on its own.  Before its running requests take a token,
             * a decoder whose tokens would pass its capacity preempts its
             * most recently admitted request (which loses its tokens and
             * goes to the head of the waiting queue) until they fit, but
             * never its last one.  Requests reaching their true length
             * complete.  On every step but the dispatch step s the queue
             * admits in order (preempted requests first, the latest on top)
             * while used + p + U <= capacity, the first misfit blocking. */
            for (int64_t t = prev_s + 1; t <= s; ++t) {
                for (int32_t k = 0; k < D; ++k) {
                    int64_t tok = 0, n = 0;
                    for (int64_t r = L.head[k]; r >= 0; r = L.next[r]) {
                        tok += (int64_t)prompt[r] + g[r];
                        ++n;
                    }
                    while (n > 1 && tok + n > capv[k]) {
                        int64_t r = L.tail[k];
                        run_unlink(&L, k, r);
                        tok -= (int64_t)prompt[r] + g[r];
                        --n;
                        st[r] = ST_WAITING;
                        g[r] = 0;
                        L.pnext[r] = L.ptop[k];
                        L.ptop[k] = r;
                        dst[4 * k + 3] += 1;
                    }
                    for (int64_t r = L.head[k], nx; r >= 0; r = nx) {
                        nx = L.next[r];
                        g[r] += 1;
                        if (g[r] == true_len[r]) {
                            run_unlink(&L, k, r);
                            st[r] = ST_DONE;
                            done[ndone].step = t;
                            done[ndone].id = r;
                            ++ndone;
                        }
                    }
                    if (t == s)
                        continue;
                    int64_t u = 0;
                    for (int64_t r = L.head[k]; r >= 0; r = L.next[r])
                        u += held_tokens(cfg->accounting, prompt[r], g[r], res_u[r]);
                    for (;;) {
                        int from_stack = L.ptop[k] >= 0;
                        if (!from_stack && L.qhead[k] >= L.qend[k])
                            break;
                        int64_t r = from_stack ? L.ptop[k] : wid[wperm[L.qhead[k]]];
                        if (u + prompt[r] + (int64_t)U[r] > capv[k])
                            break;
                        if (from_stack)
                            L.ptop[k] = L.pnext[r];
                        else
                            L.qhead[k] += 1;
                        st[r] = ST_RUNNING;
                        g[r] = 0;
                        res_u[r] = U[r];
                        u += admit_tokens(cfg->accounting, prompt[r], U[r]);
                        run_append(&L, k, r);
                        ++admitted;
                        dst[4 * k + 2] += 1;
                    }
                    /* requests waiting at decoder k through step t */
                    int64_t wq = L.qend[k] - L.qhead[k];
                    for (int64_t r = L.ptop[k]; r >= 0; r = L.pnext[r])
                        ++wq;
                    dst[4 * k] += wq;
                }
            }
        }
        for (int32_t k = 0; k < D; ++k) {
            used[k] = 0;
            occ[k] = 0;
            nreq[k] = 0;
        }
        {
            int64_t w = 0;
            for (int64_t a = 0; a < nact; ++a) {
                int64_t id = act[a];
                if (st[id] == ST_DONE)
                    continue;
                act[w++] = id;
                nreq[dec[id]] += 1; /* requests in the system (least requests) */
                if (st[id] == ST_RUNNING) {
                    /* tokens held; and what admission counts for the request
                     * (App. C: the prompt's KV once transferred, plus the
                     * output reserved at its bound until generation ends --
                     * or, without the staged release, the prompt's
                     * reservation as well) */
                    occ[dec[id]] += (int64_t)prompt[id] + g[id];
                    used[dec[id]] += held_tokens(cfg->accounting, prompt[id], g[id], res_u[id]);
                }
            }
            nact = w;
        }
        int64_t overflow = 0;
        for (int32_t k = 0; k < D; ++k) {
            overflow += occ[k] > capv[k];
            dst[4 * k + 1] += occ[k] > capv[k];
        }

        /* 2. Sliding calibration window: the most recent completions,
         *    ordered by (completion step, request id) (Sec. 3.2). */
        qsort(done, (size_t)ndone, sizeof(completion), cmp_completion);
        for (int64_t c = 0; c < ndone; ++c) {
            int64_t id = done[c].id;
            int64_t slot = (win_head + win_len) % Wn;
            if (win_len == Wn) {
                slot = win_head;
                win_head = (win_head + 1) % Wn;
            } else {
                ++win_len;
            }
            win_true[slot] = true_len[id];
            win_pred[slot] = pred[id];
        }

        /* 3. Calibrate; an unbounded quantile means the bound is unavailable
         *    and the batch falls back to round robin (Alg. 1). */
        int64_t q = 0;
        int cs = oracle_calibrate(win_true, win_pred, win_len, cfg->alpha_ppm, &q);
        int rr = 0;
        if (cs == ORACLE_E_UNBOUNDED) {
            rr = 1;
            q = 0;
        } else if (cs != ORACLE_OK) {
            status = cs;
            goto out;
        }
        q_out[b] = rr ? -1 : (int32_t)q;

        /* 4. The requests dispatched at s: the batch joins the arrived ones
         *    not yet dispatched; those whose bound is available go to the
         *    dispatch policy, those that waited beta steps past arrival
         *    without one (or are left at the last dispatch step) go round
         *    robin (Sec. 3.3, the timeout; App. D), the rest wait. */
        for (int64_t i = lo; i < hi; ++i)
            pend[npend++] = i;
        int64_t nc = 0, keep = 0, nto = 0;
        for (int64_t x = 0; x < npend; ++x) {
            int64_t id = pend[x];
            int avail = !defer || arrival_ms[id] + pred_delay[id] <= s;
            int timed_out = !avail && (arrival_ms[id] + cfg->beta <= s || b == nb - 1);
            if (avail) {
                cid[nc++] = id;
            } else if (timed_out) {
                /* round robin without a bound: projected to the horizon
                 * until its prediction arrives */
                choice_out[id] = (int32_t)(id % D);
                st[id] = ST_WAITING;
                dec[id] = (int32_t)(id % D);
                disp[id] = s;
                g[id] = 0;
                U[id] = H;
                act[nact++] = id;
                nreq[id % D] += 1;
                ++nto;
            } else {
                pend[keep++] = id;
            }
        }
        npend = keep;

        /*    Bounds for every request in the system (the horizon while its
         *    prediction is not in yet) and for the policy's candidates. */
        for (int64_t a = 0; a < nact; ++a) {
            int64_t id = act[a];
            int32_t u = H;
            if ((!defer || arrival_ms[id] + pred_delay[id] <= s) &&
                oracle_bound(&pred[id], 1, q, &u) != ORACLE_OK)
                status = ORACLE_E_RANGE;
            U[id] = u;
        }
        for (int64_t c = 0; c < nc; ++c) {
            cp[c] = prompt[cid[c]];
            if (oracle_bound(&pred[cid[c]], 1, q, &cU[c]) != ORACLE_OK)
                status = ORACLE_E_RANGE;
        }

        /* 5. Dispatch the candidates. */
        if (!rr && cfg->dispatch == 3) {
            /* least requests: the decoder with the fewest requests in the
             * system, the candidates counted as they are dispatched */
            for (int64_t c = 0; c < nc; ++c) {
                int32_t best = 0;
                for (int32_t k = 1; k < D; ++k)
                    if (nreq[k] < nreq[best])
                        best = k;
                cch[c] = best;
                nreq[best] += 1;
            }
        } else if (!rr && cfg->dispatch != 2) {
            /* residents of each decoder: running (g) and waiting (g = 0) */
            int64_t R = 0;
            for (int32_t k = 0; k < D; ++k) {
                off[k] = R;
                Q[k] = 0;
                for (int64_t a = 0; a < nact; ++a) {
                    int64_t id = act[a];
                    if (dec[id] != k)
                        continue;
                    rp[R] = prompt[id];
                    rg[R] = st[id] == ST_RUNNING ? g[id] : 0;
                    rU[R] = U[id];
                    ++R;
                    Q[k] += st[id] == ST_WAITING;
                }
            }
            off[D] = R;
            int os = oracle_occupancy(D, H, off, R, rp, rg, rU, K);
            if (os != ORACLE_OK)
                status = os;
            int ds = dispatch_horizon(1, cfg->dispatch == 1, D, H, K, capv, Q,
                                      nc, cp, cU, cch, hr);
            if (ds != ORACLE_OK)
                status = ds;
        } else {
            for (int64_t c = 0; c < nc; ++c)
                cch[c] = (int32_t)(cid[c] % D);
        }

        /* 6. The candidates join the chosen decoders' waiting queues. */
        for (int64_t c = 0; c < nc; ++c) {
            int64_t i = cid[c];
            choice_out[i] = cch[c];
            st[i] = ST_WAITING;
            dec[i] = cch[c];
            disp[i] = s;
            g[i] = 0;
            U[i] = cU[c];
            act[nact++] = i;
        }
        (void)nto;

        /* 7. Local order of every waiting queue. */
        int64_t nw = 0;
        for (int64_t a = 0; a < nact; ++a) {
            int64_t id = act[a];
            if (st[id] != ST_WAITING)
                continue;
            int64_t w = s - disp[id];
            wid[nw] = id;
            wdec[nw] = dec[id];
            wU[nw] = U[id];
            wwait[nw] = (int32_t)(w > I32_MAX ? I32_MAX : w);
            warr[nw] = (int32_t)id;
            ++nw;
        }
        /* FCFS promotes every entry: arrival order alone */
        int ls = oracle_order_local(nw, D, wdec, wU, wwait, warr,
                                    cfg->local == 1 ? -1 : cfg->max_wait, wperm, seg);
        if (ls != ORACLE_OK) {
            status = ls;
            goto out;
        }

        /* 8. Admission in queue order while the current occupancy plus the
         *    request's bounded demand fits, Eq. (admission) with the
         *    calibrated bound standing in for the unknown output length;
         *    the first misfit blocks the rest of its queue. */
        int64_t admitted8 = 0;
        for (int32_t k = 0; k < D; ++k) {
            int64_t x = seg[k];
            for (; x < seg[k + 1]; ++x) {
                int64_t id = wid[wperm[x]];
                int64_t demand = (int64_t)prompt[id] + U[id];
                if (used[k] + demand > capv[k])
                    break;
                st[id] = ST_RUNNING;
                g[id] = 0;
                res_u[id] = U[id];
                used[k] += admit_tokens(cfg->accounting, prompt[id], U[id]);
                ++admitted8;
                dst[4 * k + 2] += 1;
                if (cfg->per_step)
                    run_append(&L, k, id);
            }
            int64_t left = seg[k + 1] - x;
            if (cfg->per_step) {
                /* the rest of the queue, in this order, until the next
                 * dispatch step; preempted requests have all been ordered */
                L.qhead[k] = x;
                L.qend[k] = seg[k + 1];
                L.ptop[k] = -1;
                if (b + 1 < nb)
                    dst[4 * k] += left; /* waiting through step s */
            } else {
                /* the waiting queue holds until the next batch's dispatch step */
                int64_t s_next = b + 1 < nb ? arrival_ms[((b + 2) * Bsz < N ? (b + 2) * Bsz : N) - 1] : s;
                dst[4 * k] += left * (s_next - s);
            }
        }
        stats_out[4 * b + 0] = ndone;
        stats_out[4 * b + 1] = admitted + admitted8;
        stats_out[4 * b + 2] = nw - admitted8;
        stats_out[4 * b + 3] = overflow;
        prev_s = s;
    }
    if (dec_stats_out != NULL)
        for (int64_t i = 0; i < (int64_t)D * 4; ++i)
            dec_stats_out[i] = dst[i];

out:
    free(st); free(g); free(dec); free(U); free(disp); free(act); free(done);
    free(win_true); free(win_pred); free(K); free(capv); free(Q); free(off);
    free(used); free(seg); free(rp); free(rg); free(rU); free(wid); free(wdec);
    free(wU); free(wwait); free(warr); free(wperm); free(cid); free(cp); free(cU);
    free(cch); free(hr); free(pend); free(res_u); free(occ); free(nreq); free(dst);
    free(L.next); free(L.prev); free(L.pnext); free(L.head); free(L.tail);
    free(L.ptop); free(L.qhead); free(L.qend);
    return status;
}
