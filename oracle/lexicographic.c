/*
 * Oracle for tiers 3 and 4 of the lexicographic objective and the goodput
 * gap.
 *
 * TEST INFRASTRUCTURE ONLY (see fs_oracle.h).
 *
 * Section 3: the objective is lexicographic: (1) critical floors, (2) max
 * min_i r_i, (3) maximise total served goodput, (4) minimise fragmentation.
 * Tiers 1-2 are or_solve_literal / or_solve_frontier (threshold rule, t*).
 * This file adds, among the allocations that keep tiers 1-2 optimal:
 *
 *   tier 3: the largest goodput sum_i x_i with x_i = min(lambda_i, n c)
 *     (Eqs. 2 and 4), each class's term taken in fixed point,
 *     rint(x_i 2^20) (units of 2^-20 req/s), so that sums are exact;
 *   tier 4: the fewest GPUs in use (no GPU held without adding goodput),
 *     then, class by class in index order, the tie rules of the threshold
 *     solver (lower TP, fewer replicas, larger capacity, lower bin).
 *
 * Keeping tiers 1-2 optimal: when t* > 0 every class must reach
 * r_i >= max(t*, delta_i); when t* = 0 and the floors are met, critical
 * classes must reach their floors and every other class may take any
 * option or none; when the floors cannot be met nothing is allocated.
 *
 * The search is a dynamic programme over classes (from the last) and GPUs
 * left, on one row per (class, TP): a larger capacity never lowers
 * goodput or fulfilment at equal cost, so the best SLO-feasible bin of a row
 * (largest capacity, then lowest bin) carries every useful option; replica
 * counts beyond the first that serves the whole demand add GPUs and no
 * goodput and are never chosen. The tests hold it to brute-force
 * enumeration of every allocation (tests/brute.py) and to the paper's
 * Table 3 (allocations and goodput at 0.7x, 1.0x and 1.3x demand).
 *
 * The goodput gap (the second curve of Fig. 4a, and the third stage of the
 * stage-wise certificate of Section 4.2): |GP(A+) - GP(A-)| / sum_i lambda_i.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "fs_oracle.h"

static const int TPD[OR_T] = {1, 2, 4, 8};

int64_t or_goodput_fx(int n, float c, float lam)
{
    float served = (float)n * c;
    float x = served < lam ? served : lam;
    return llrintf(x * 0x1p20f);
}

static float floor_i(const or_problem *p, int i) { return p->floor ? p->floor[i] : 0.0f; }

typedef struct {
    int64_t gp;   /* goodput, 2^-20 req/s */
    int gpus;
    int ok;       /* reachable */
} dpcell;

/* a better than b: more goodput, then fewer GPUs */
static int dp_better(int64_t gpa, int gpusa, int64_t gpb, int gpusb)
{
    if (gpa != gpb) return gpa > gpb;
    return gpusa < gpusb;
}

int or_solve_lex(const or_problem *p, const float *cap, const float *tail, int solver,
                 or_alloc *out, int64_t *goodput_fx)
{
    or_alloc a;
    int rc = solver == 0 ? or_solve_literal(p, cap, tail, &a) : or_solve_frontier(p, cap, tail, &a);
    if (rc) return rc;
    *out = a;
    *goodput_fx = 0;
    if (!a.floors_met) return 0;  /* tier 1 cannot hold: nothing is allocated */
    const int K = p->K, B = p->B, G = p->G;
    const float tstar = a.t_star;

    /* best SLO-feasible bin per (class, TP) row */
    float C[OR_KMAX][OR_T];
    int bb[OR_KMAX][OR_T];
    for (int i = 0; i < K; ++i)
        for (int j = 0; j < OR_T; ++j) {
            bb[i][j] = -1;
            C[i][j] = 0.0f;
            for (int b = 0; b < B; ++b) {
                int cell = (i * OR_T + j) * B + b;
                if (!(tail[cell] <= p->slo[i])) continue;
                if (bb[i][j] < 0 || cap[cell] > C[i][j]) {
                    C[i][j] = cap[cell];
                    bb[i][j] = b;
                }
            }
        }
    /* per class: the fulfilment it must reach, and whether it may stay empty */
    float T[OR_KMAX];
    int may_empty[OR_KMAX];
    for (int i = 0; i < K; ++i) {
        float d = floor_i(p, i);
        if (tstar > 0.0f) {
            T[i] = tstar > d ? tstar : d;
            may_empty[i] = 0;
        } else {
            T[i] = d;
            may_empty[i] = !(d > 0.0f);
        }
    }

    /* suffix programme: S[i][g] = best (goodput, GPUs) of classes i..K-1 within g GPUs */
    size_t W = (size_t)G + 1;
    dpcell *S = (dpcell *)calloc((size_t)(K + 1) * W, sizeof(dpcell));
    if (!S) return -2;
    for (size_t g = 0; g < W; ++g) S[(size_t)K * W + g].ok = 1;
    for (int i = K - 1; i >= 0; --i) {
        dpcell *cur = S + (size_t)i * W, *nxt = S + (size_t)(i + 1) * W;
        for (int g = 0; g <= G; ++g) {
            dpcell best = {0, 0, 0};
            if (may_empty[i] && nxt[g].ok) best = nxt[g];
            for (int j = 0; j < OR_T; ++j) {
                if (bb[i][j] < 0) continue;
                for (int n = 1; n <= G / TPD[j] && n * TPD[j] <= g; ++n) {
                    float f = or_fulfil(n, C[i][j], p->demand[i]);
                    if (T[i] > 0.0f && !(f >= T[i])) continue;
                    int cost = n * TPD[j];
                    if (!nxt[g - cost].ok) continue;
                    int64_t v = or_goodput_fx(n, C[i][j], p->demand[i]) + nxt[g - cost].gp;
                    int u = cost + nxt[g - cost].gpus;
                    if (!best.ok || dp_better(v, u, best.gp, best.gpus)) {
                        best.gp = v;
                        best.gpus = u;
                        best.ok = 1;
                    }
                    /* past the first count serving the whole demand: same goodput, more GPUs */
                    if (!((float)n * C[i][j] < p->demand[i])) break;
                }
            }
            cur[g] = best;
        }
    }
    if (!S[G].ok) {  /* cannot happen: the tier-2 allocation is feasible */
        free(S);
        return -3;
    }
    *goodput_fx = S[G].gp;

    /* forward: class by class, the preferred option that keeps the optimum */
    int left = G, total = 0;
    for (int i = 0; i < K; ++i) {
        const dpcell target = S[(size_t)i * W + left];
        const dpcell *nxt = S + (size_t)(i + 1) * W;
        int cj = -1, cn = 0;
        if (may_empty[i] && nxt[left].ok && nxt[left].gp == target.gp && nxt[left].gpus == target.gpus) {
            cj = -1;  /* no replicas: preferred when it keeps the optimum */
        } else {
            for (int j = 0; j < OR_T && cj < 0; ++j) {
                if (bb[i][j] < 0) continue;
                for (int n = 1; n <= G / TPD[j] && n * TPD[j] <= left; ++n) {
                    float f = or_fulfil(n, C[i][j], p->demand[i]);
                    if (T[i] > 0.0f && !(f >= T[i])) continue;
                    int cost = n * TPD[j];
                    if (!nxt[left - cost].ok) continue;
                    if (or_goodput_fx(n, C[i][j], p->demand[i]) + nxt[left - cost].gp == target.gp &&
                        cost + nxt[left - cost].gpus == target.gpus) {
                        cj = j;
                        cn = n;
                        break;
                    }
                }
            }
        }
        out->tp[i] = cj >= 0 ? TPD[cj] : 0;
        out->bin[i] = cj >= 0 ? bb[i][cj] : -1;
        out->replicas[i] = cn;
        out->fulfil[i] = cj >= 0 ? or_fulfil(cn, C[i][cj], p->demand[i]) : 0.0f;
        if (cj >= 0) {
            left -= cn * TPD[cj];
            total += cn * TPD[cj];
        }
    }
    out->total_gpus = total;
    free(S);
    return 0;
}

static double demand_sum(const or_problem *p)
{
    double s = 0.0;
    for (int i = 0; i < p->K; ++i) s += (double)p->demand[i];
    return s;
}

static int64_t abs64(int64_t x) { return x < 0 ? -x : x; }

int or_base_gap_lex(const or_problem *p, const float *cap_lo, const float *cap_hi,
                    const float *tail_lo, const float *tail_hi, int solver,
                    or_alloc *minus, or_alloc *plus, int64_t *gp_minus, int64_t *gp_plus,
                    float *gamma_mm, double *gamma_gp)
{
    int rc = or_solve_lex(p, cap_lo, tail_hi, solver, minus, gp_minus);
    if (!rc) rc = or_solve_lex(p, cap_hi, tail_lo, solver, plus, gp_plus);
    if (rc) return rc;
    *gamma_mm = plus->t_star - minus->t_star;
    *gamma_gp = ((double)abs64(*gp_plus - *gp_minus) * 0x1p-20) / demand_sum(p);
    return 0;
}

/*
 * Section 4.2, stage-wise: certified infeasible when even A+ misses a
 * critical floor; certified feasible when A- meets the floors, every cell
 * A- commits replicas to (its tier-4 allocation) is revealed, and both the
 * max-min gap and the goodput gap are at most eps; otherwise undecided.
 */
int or_certificate_lex(const or_problem *p, const float *cap_lo, const float *cap_hi,
                       const float *tail_lo, const float *tail_hi, const uint8_t *revealed,
                       float eps, int solver, int *state, float *gamma_mm, double *gamma_gp)
{
    or_alloc am, ap;
    int64_t gm, gpl;
    int rc = or_base_gap_lex(p, cap_lo, cap_hi, tail_lo, tail_hi, solver, &am, &ap, &gm, &gpl,
                             gamma_mm, gamma_gp);
    if (rc) return rc;
    int known = 1;
    for (int i = 0; i < p->K; ++i) {
        if (am.replicas[i] <= 0) continue;
        int j = 0;
        while (j < OR_T && TPD[j] != am.tp[i]) ++j;
        if (!revealed[(i * OR_T + j) * p->B + am.bin[i]]) known = 0;
    }
    if (!ap.floors_met) *state = 2;
    else *state = (am.floors_met && known && *gamma_mm <= eps && *gamma_gp <= (double)eps) ? 1 : 0;
    return 0;
}

/*
 * The goodput stage of Section 4.3's score: for every candidate e, outcome o
 * and sample s, the same draw and realisations as or_score (the problem's
 * prior included), both solved to tier 4, and the scenario's goodput gap
 * |GP(A+') - GP(A-')| summed in int64 (units of 2^-20 req/s). Then
 * E[Gamma_gp,t+1 | e] = sum / (O S) 2^-20 / sum_i lambda_i, the score
 * Gamma_gp,t - E (fixed point: |GP+ - GP-| O S - sum) and the argmax with
 * the same tie rules. sum_i lambda_i 2^42 must stay below 2^63.
 */
int or_score_goodput(const or_problem *p, const float *cap_lo, const float *cap_hi,
                     const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                     uint64_t seed, uint32_t stream_id, uint32_t round,
                     int n_cand, const int32_t *cand, int O, int S, int solver,
                     int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed,
                     int64_t *gamma_fx, double *gamma_gp, int32_t *best)
{
    if (n_cand < 0 || O < 1 || S < 1 || Q % O != 0) return -1;
    if ((int64_t)O * S > ((int64_t)1 << 22)) return -1;
    const int cells = p->K * OR_T * p->B;
    for (int e = 0; e < n_cand; ++e)
        if (cand[e] < 0 || cand[e] >= cells) return -1;
    const double lam_sum = demand_sum(p);
    or_alloc am, ap;
    int64_t gm, gpl;
    float gmm;
    double ggp;
    int rc = or_base_gap_lex(p, cap_lo, cap_hi, tail_lo, tail_hi, solver, &am, &ap, &gm, &gpl, &gmm, &ggp);
    if (rc) return rc;
    const int64_t g_t = abs64(gpl - gm);
    if (gamma_fx) *gamma_fx = g_t;
    if (gamma_gp) *gamma_gp = ggp;
    const int64_t n = (int64_t)O * S;

    float *cm = (float *)malloc(sizeof(float) * cells * 4);
    if (!cm) return -2;
    float *tm = cm + cells, *cp = cm + 2 * cells, *tp = cm + 3 * cells;
    memcpy(cm, cap_lo, sizeof(float) * cells);
    memcpy(tm, tail_hi, sizeof(float) * cells);
    memcpy(cp, cap_hi, sizeof(float) * cells);
    memcpy(tp, tail_lo, sizeof(float) * cells);
    int best_e = -1;
    int64_t best_sc = 0;
    for (int e = 0; e < n_cand; ++e) {
        const int32_t cell = cand[e];
        const int first = (cell / p->B) * p->B;
        int64_t tot = 0;
        for (int o = 0; o < O; ++o) {
            int64_t acc = 0;
            for (int s = 0; s < S; ++s) {
                int32_t kc, kl;
                or_draw_index(seed, stream_id, round, cell, Q, O, o, s, &kc, &kl);
                float cy = or_map(cap_lo[cell], cap_hi[cell], qn[kc]);
                float ly = or_map(tail_lo[cell], tail_hi[cell], qn[kl]);
                for (int x = first; x < first + p->B; ++x) {
                    cm[x] = cap_lo[x]; cp[x] = cap_hi[x];
                    tp[x] = tail_lo[x]; tm[x] = tail_hi[x];
                }
                or_refit(p, p->prior, cell, cy, ly, cm, cp, tp, tm);
                rc = or_solve_lex(p, cm, tm, solver, &am, &gm);
                if (!rc) rc = or_solve_lex(p, cp, tp, solver, &ap, &gpl);
                if (rc) { free(cm); return rc; }
                acc += abs64(gpl - gm);
            }
            if (sum_eo) sum_eo[(size_t)e * O + o] = acc;
            tot += acc;
        }
        for (int x = first; x < first + p->B; ++x) {
            cm[x] = cap_lo[x]; cp[x] = cap_hi[x];
            tp[x] = tail_lo[x]; tm[x] = tail_hi[x];
        }
        int64_t sc = g_t * n - tot;
        if (gap) gap[e] = ((double)tot * 0x1p-20) / (double)n / lam_sum;
        if (score) score[e] = ((double)sc * 0x1p-20) / (double)n / lam_sum;
        if (score_fixed) score_fixed[e] = sc;
        int j = (cell / p->B) % OR_T;
        if (best_e < 0 || sc > best_sc || (sc == best_sc && j < (cand[best_e] / p->B) % OR_T)) {
            best_e = e;
            best_sc = sc;
        }
    }
    free(cm);
    if (best) *best = best_e >= 0 ? cand[best_e] : -1;
    return 0;
}
