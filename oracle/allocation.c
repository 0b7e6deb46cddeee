/*
 * Oracle allocation solvers.
 *
 * TEST INFRASTRUCTURE ONLY (see fs_oracle.h).
 *
 * The allocation model is Section 3, Eqs. 1-5: class i picks one
 * homogeneous configuration q = (TP degree tau, load bin b) (Eq. 1) and an
 * integer replica count n; it serves x_i <= min(lambda_i, n c_iq)
 * (Eqs. 2, 4); the replicas use n tau GPUs and all classes together use at
 * most G (Eq. 3); a configuration whose tail exceeds the class SLO cannot
 * be chosen (Eq. 5). The objective's tier 2 is max_i-min r_i with
 * r_i = x_i / lambda_i. The replica cap M of Eq. 1 is read as floor(G/tau).
 *
 * Tier 2 is solved with the threshold rule: for a threshold t, each class
 * takes its cheapest SLO-feasible option whose fulfilment is at least t;
 * t* is the largest option fulfilment whose cheapest covers fit in G.
 * Ties between options of equal GPU cost go to the lower TP degree, then
 * to fewer replicas, then to the larger capacity, then to the lower bin.
 * If no positive threshold fits (including when some class has no
 * SLO-feasible option at all), t* = 0 and every class gets nothing.
 * The success-rate gate of Eq. 5 is taken as satisfied (no success data).
 *
 * Tier 1 (critical floors): a critical class i (delta_i > 0) must reach
 * r_i >= delta_i whenever that is possible. Its options below the floor are
 * therefore not options at all; tier 2 is solved on what remains (the
 * threshold rule then gives every class the cheapest cover of
 * max(t, delta_i)). The floors are met when every critical class has an
 * option at or above its floor and their cheapest such options fit in G
 * together (the other classes may stay empty). When no positive threshold
 * fits but the floors are met, each critical class still gets its cheapest
 * option at or above its floor (same tie rules) and the others nothing; when
 * the floors cannot be met, t* = 0 (no class can be served at a positive
 * threshold while they hold) and every class gets nothing.
 */
#include <stdlib.h>
#include <string.h>
#include "fs_oracle.h"

static const int OR_TP[OR_T] = {1, 2, 4, 8};

/* f(n, c) = min(1, (n c) / lambda): r_i of Section 3 with x_i = min(lambda, n c). */
float or_fulfil(int n, float c, float lam)
{
    float served = (float)n * c;
    float r = served / lam;
    return r > 1.0f ? 1.0f : r;
}

static int check_problem(const or_problem *p)
{
    if (!p || p->K < 1 || p->K > OR_KMAX || p->B < 1 || p->G < 1) return -1;
    for (int i = 0; i < p->K; ++i) {
        if (!(p->demand[i] > 0.0f)) return -1;
        if (p->floor && !(p->floor[i] >= 0.0f && p->floor[i] <= 1.0f)) return -1;
    }
    return 0;
}

/* delta_i, the fulfilment floor of class i (0: not critical). */
static float floor_of(const or_problem *p, int i)
{
    return p->floor ? p->floor[i] : 0.0f;
}

static void empty_alloc(const or_problem *p, uint64_t mask, or_alloc *out)
{
    memset(out, 0, sizeof(*out));
    out->has_option_mask = mask;
    for (int i = 0; i < p->K; ++i) {
        out->tp[i] = 0;
        out->bin[i] = -1;
        out->replicas[i] = 0;
        out->fulfil[i] = 0.0f;
    }
}

typedef struct {
    int cls, j, b, n, cost;
    float f, cap;
} option;

/* a strictly preferred to b (both cover the threshold). */
static int prefer(const option *a, const option *b)
{
    if (a->cost != b->cost) return a->cost < b->cost;
    if (a->j != b->j) return a->j < b->j;
    if (a->n != b->n) return a->n < b->n;
    if (a->cap != b->cap) return a->cap > b->cap;
    return a->b < b->b;
}

static int cmp_desc(const void *x, const void *y)
{
    float a = *(const float *)x, b = *(const float *)y;
    return (a < b) - (a > b);
}

/*
 * Literal solver: enumerate every option (tau, b, n) of every class, take
 * the set of their fulfilment values as thresholds, and sweep them from the
 * largest down; the first threshold whose cheapest per-class covers fit in
 * G is t*.
 */
int or_solve_literal(const or_problem *p, const float *cap, const float *tail, or_alloc *out)
{
    if (check_problem(p)) return -1;
    const int K = p->K, B = p->B, G = p->G;
    size_t max_opt = 0;
    for (int j = 0; j < OR_T; ++j) max_opt += (size_t)K * B * (G / OR_TP[j]);
    option *opt = (option *)malloc((max_opt + 1) * sizeof(option));
    float *theta = (float *)malloc((max_opt + 1) * sizeof(float));
    int *first = (int *)malloc((K + 1) * sizeof(int));
    if (!opt || !theta || !first) {
        free(opt); free(theta); free(first);
        return -2;
    }
    size_t n_opt = 0, n_theta = 0;
    uint64_t mask = 0;
    for (int i = 0; i < K; ++i) {
        first[i] = (int)n_opt;
        for (int j = 0; j < OR_T; ++j) {
            int tau = OR_TP[j];
            int M = G / tau;
            for (int b = 0; b < B; ++b) {
                int cell = (i * OR_T + j) * B + b;
                if (!(tail[cell] <= p->slo[i])) continue;   /* Eq. 5 */
                mask |= (uint64_t)1 << i;
                for (int n = 1; n <= M; ++n) {
                    option o;
                    o.cls = i; o.j = j; o.b = b; o.n = n;
                    o.cost = n * tau;
                    o.cap = cap[cell];
                    o.f = or_fulfil(n, cap[cell], p->demand[i]);
                    if (o.f < floor_of(p, i)) continue;      /* tier 1: below the floor */
                    opt[n_opt++] = o;
                    if (o.f > 0.0f) theta[n_theta++] = o.f;
                }
            }
        }
    }
    first[K] = (int)n_opt;
    qsort(theta, n_theta, sizeof(float), cmp_desc);

    int found = 0;
    option chosen[OR_KMAX];
    for (size_t q = 0; q < n_theta && !found; ++q) {
        if (q > 0 && theta[q] == theta[q - 1]) continue;   /* distinct thresholds */
        float t = theta[q];
        long total = 0;
        int all = 1;
        for (int i = 0; i < K && all; ++i) {
            int best = -1;
            for (int k = first[i]; k < first[i + 1]; ++k) {
                if (opt[k].f >= t && (best < 0 || prefer(&opt[k], &opt[best]))) best = k;
            }
            if (best < 0) {
                all = 0;
            } else {
                chosen[i] = opt[best];
                total += opt[best].cost;
            }
        }
        if (all && total <= G) {
            found = 1;
            empty_alloc(p, mask, out);
            out->t_star = t;
            out->total_gpus = (int32_t)total;
            out->ok = 1;
            out->floors_met = 1;
            for (int i = 0; i < K; ++i) {
                out->tp[i] = OR_TP[chosen[i].j];
                out->bin[i] = chosen[i].b;
                out->replicas[i] = chosen[i].n;
                out->fulfil[i] = chosen[i].f;
            }
        }
    }
    if (!found) {
        /* tier 1 alone: each critical class's preferred option (all of its
         * remaining options are at or above its floor) */
        long total = 0;
        int met = 1;
        for (int i = 0; i < K; ++i) {
            chosen[i].n = 0;
            if (floor_of(p, i) <= 0.0f) continue;
            int best = -1;
            for (int k = first[i]; k < first[i + 1]; ++k)
                if (best < 0 || prefer(&opt[k], &opt[best])) best = k;
            if (best < 0) {
                met = 0;
            } else {
                chosen[i] = opt[best];
                total += opt[best].cost;
            }
        }
        if (total > G) met = 0;
        empty_alloc(p, mask, out);
        out->floors_met = met;
        if (met) {
            out->total_gpus = (int32_t)total;
            for (int i = 0; i < K; ++i) {
                if (floor_of(p, i) <= 0.0f) continue;
                out->tp[i] = OR_TP[chosen[i].j];
                out->bin[i] = chosen[i].b;
                out->replicas[i] = chosen[i].n;
                out->fulfil[i] = chosen[i].f;
            }
        }
    }
    free(opt); free(theta); free(first);
    return 0;
}

/* Smallest n in [1, M] with f(n, c) >= t, or 0 if none (f is nondecreasing in n). */
static int min_replicas(float t, float c, float lam, int M)
{
    if (M < 1 || or_fulfil(M, c, lam) < t) return 0;
    int lo = 1, hi = M;
    while (lo < hi) {
        int mid = lo + (hi - lo) / 2;
        if (or_fulfil(mid, c, lam) >= t) hi = mid; else lo = mid + 1;
    }
    return lo;
}

/* Cheapest cover of threshold t by class i over its rows (best bin of each
 * TP degree): its GPU cost, or -1 if no row covers t; equal costs keep the
 * lower TP. */
static int cheapest_cover(const or_problem *p, const float *Ci, const int *bi, int i, float t,
                          int *j_out, int *n_out)
{
    int best_cost = -1;
    *j_out = -1;
    *n_out = 0;
    for (int j = 0; j < OR_T; ++j) {
        if (bi[j] < 0) continue;
        int n = min_replicas(t, Ci[j], p->demand[i], p->G / OR_TP[j]);
        if (n == 0) continue;
        int cost = n * OR_TP[j];
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            *j_out = j;
            *n_out = n;
        }
    }
    return best_cost;
}

/*
 * Frontier solver: the same threshold rule, evaluated on one row per
 * (class, TP): for a fixed (tau, n) a larger capacity never lowers the
 * fulfilment, so the best SLO-feasible bin of the row (largest capacity,
 * then lowest bin) is the one the literal tie rule picks. Thresholds are
 * the row values; the sweep runs from the largest down. Pinned against
 * or_solve_literal and brute force in the tests.
 */
int or_solve_frontier(const or_problem *p, const float *cap, const float *tail, or_alloc *out)
{
    if (check_problem(p)) return -1;
    const int K = p->K, B = p->B, G = p->G;
    float C[OR_KMAX][OR_T];
    int bstar[OR_KMAX][OR_T];
    uint64_t mask = 0;
    size_t max_theta = 0;
    for (int i = 0; i < K; ++i) {
        for (int j = 0; j < OR_T; ++j) {
            bstar[i][j] = -1;
            C[i][j] = 0.0f;
            for (int b = 0; b < B; ++b) {
                int cell = (i * OR_T + j) * B + b;
                if (!(tail[cell] <= p->slo[i])) continue;
                if (bstar[i][j] < 0 || cap[cell] > C[i][j]) {
                    C[i][j] = cap[cell];
                    bstar[i][j] = b;
                }
            }
            if (bstar[i][j] >= 0) {
                mask |= (uint64_t)1 << i;
                max_theta += (size_t)(G / OR_TP[j]);
            }
        }
    }
    float *theta = (float *)malloc((max_theta + 1) * sizeof(float));
    if (!theta) return -2;
    size_t n_theta = 0;
    for (int i = 0; i < K; ++i)
        for (int j = 0; j < OR_T; ++j) {
            if (bstar[i][j] < 0) continue;
            int M = G / OR_TP[j];
            for (int n = 1; n <= M; ++n) {
                float f = or_fulfil(n, C[i][j], p->demand[i]);
                if (f > 0.0f && f >= floor_of(p, i)) theta[n_theta++] = f;
            }
        }
    qsort(theta, n_theta, sizeof(float), cmp_desc);

    int found = 0;
    int cj[OR_KMAX], cn[OR_KMAX];
    for (size_t q = 0; q < n_theta && !found; ++q) {
        if (q > 0 && theta[q] == theta[q - 1]) continue;
        float t = theta[q];
        long total = 0;
        int all = 1;
        for (int i = 0; i < K && all; ++i) {
            /* class i must cover max(t, delta_i) */
            float ti = t > floor_of(p, i) ? t : floor_of(p, i);
            int cost = cheapest_cover(p, C[i], bstar[i], i, ti, &cj[i], &cn[i]);
            if (cost < 0) all = 0; else total += cost;
        }
        if (all && total <= G) {
            found = 1;
            empty_alloc(p, mask, out);
            out->t_star = t;
            out->total_gpus = (int32_t)total;
            out->ok = 1;
            out->floors_met = 1;
            for (int i = 0; i < K; ++i) {
                int j = cj[i];
                out->tp[i] = OR_TP[j];
                out->bin[i] = bstar[i][j];
                out->replicas[i] = cn[i];
                out->fulfil[i] = or_fulfil(cn[i], C[i][j], p->demand[i]);
            }
        }
    }
    if (!found) {
        /* tier 1 alone: each critical class's cheapest cover of its floor */
        long total = 0;
        int met = 1;
        for (int i = 0; i < K; ++i) {
            cn[i] = 0;
            if (floor_of(p, i) <= 0.0f) continue;
            int cost = cheapest_cover(p, C[i], bstar[i], i, floor_of(p, i), &cj[i], &cn[i]);
            if (cost < 0) met = 0; else total += cost;
        }
        if (total > G) met = 0;
        empty_alloc(p, mask, out);
        out->floors_met = met;
        if (met) {
            out->total_gpus = (int32_t)total;
            for (int i = 0; i < K; ++i) {
                if (cn[i] <= 0) continue;
                int j = cj[i];
                out->tp[i] = OR_TP[j];
                out->bin[i] = bstar[i][j];
                out->replicas[i] = cn[i];
                out->fulfil[i] = or_fulfil(cn[i], C[i][j], p->demand[i]);
            }
        }
    }
    free(theta);
    return 0;
}

/*
 * Objective of a given allocation: max-min fulfilment (tier 2) and served
 * goodput sum_i min(lambda_i, n c) (tier 3, Section 3). A class with no
 * option (tp_index < 0) or with an SLO-infeasible cell serves nothing.
 */
int or_evaluate(const or_problem *p, const float *cap, const float *tail,
                const int32_t *tp_index, const int32_t *bin, const int32_t *replicas,
                double *max_min, double *goodput)
{
    if (check_problem(p)) return -1;
    double mm = 1.0, gp = 0.0;
    long gpus = 0;
    for (int i = 0; i < p->K; ++i) {
        float f = 0.0f, x = 0.0f;
        if (tp_index[i] >= 0 && replicas[i] > 0) {
            int cell = (i * OR_T + tp_index[i]) * p->B + bin[i];
            if (tail[cell] <= p->slo[i]) {
                float served = (float)replicas[i] * cap[cell];
                x = served < p->demand[i] ? served : p->demand[i];
                f = or_fulfil(replicas[i], cap[cell], p->demand[i]);
            }
            gpus += (long)replicas[i] * OR_TP[tp_index[i]];
        }
        if ((double)f < mm) mm = f;
        gp += x;
    }
    *max_min = mm;
    *goodput = gp;
    return gpus <= p->G ? 0 : 1;
}
