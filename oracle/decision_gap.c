/*
 * Oracle decision gap, acquisition score, certificate and profiling loop.
 *
 * TEST INFRASTRUCTURE ONLY (see fs_oracle.h).
 *
 * Section 4.1: A- takes every cell at (lower capacity, upper tail), A+ at
 * (upper capacity, lower tail); both use the same G, SLO policy and
 * objective. Section 4.2: the gap is the difference of their objectives;
 * here the tier-2 objective, Gamma = t*(A+) - t*(A-) (the "max-min gap").
 * Section 4.3: score_t(e) = E[Gamma_t - Gamma_{t+1} | e]; the expectation is
 * a Monte-Carlo mean over O outcome strata x S samples. Revealing e
 * collapses its interval to the drawn point in both realisations and refits
 * the other intervals under the problem's prior (prior.c): none under the
 * revealed-only prior, the rest of e's row under the monotone prior.
 *
 * Sums are taken in fixed point: g = rint(Gamma' * 2^40) as int64, so the
 * result does not depend on summation order.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "fs_oracle.h"

static int solve(const or_problem *p, const float *cap, const float *tail, int solver, or_alloc *out)
{
    return solver == 0 ? or_solve_literal(p, cap, tail, out) : or_solve_frontier(p, cap, tail, out);
}

int or_base_gap(const or_problem *p, const float *cap_lo, const float *cap_hi,
                const float *tail_lo, const float *tail_hi, int solver,
                or_alloc *minus, or_alloc *plus, float *gamma_t)
{
    int rc = solve(p, cap_lo, tail_hi, solver, minus);
    if (rc) return rc;
    rc = solve(p, cap_hi, tail_lo, solver, plus);
    if (rc) return rc;
    *gamma_t = plus->t_star - minus->t_star;
    return 0;
}

static int cells_of(const or_problem *p) { return p->K * OR_T * p->B; }

/* The base bounds of cell's row back into the realisations' working arrays
 * (cm = cap_lo, cp = cap_hi, tp = tail_lo, tm = tail_hi). */
static void restore_row(const or_problem *p, int32_t cell, const float *cap_lo, const float *cap_hi,
                        const float *tail_lo, const float *tail_hi,
                        float *cm, float *cp, float *tp, float *tm)
{
    int first = (cell / p->B) * p->B;
    for (int x = first; x < first + p->B; ++x) {
        cm[x] = cap_lo[x]; cp[x] = cap_hi[x];
        tp[x] = tail_lo[x]; tm[x] = tail_hi[x];
    }
}

int or_scenario(const or_problem *p, const float *cap_lo, const float *cap_hi,
                const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                uint64_t seed, uint32_t stream_id, uint32_t round, int32_t cell,
                int O, int o, int s, int solver,
                float *c_y, float *l_y, or_alloc *minus, or_alloc *plus)
{
    int cells = cells_of(p);
    if (cell < 0 || cell >= cells) return -1;
    int32_t kc, kl;
    if (or_draw_index(seed, stream_id, round, cell, Q, O, o, s, &kc, &kl)) return -1;
    float cy = or_map(cap_lo[cell], cap_hi[cell], qn[kc]);
    float ly = or_map(tail_lo[cell], tail_hi[cell], qn[kl]);
    float *cm = (float *)malloc(sizeof(float) * cells * 4);
    if (!cm) return -2;
    float *tm = cm + cells, *cp = cm + 2 * cells, *tp = cm + 3 * cells;
    memcpy(cm, cap_lo, sizeof(float) * cells);
    memcpy(tm, tail_hi, sizeof(float) * cells);
    memcpy(cp, cap_hi, sizeof(float) * cells);
    memcpy(tp, tail_lo, sizeof(float) * cells);
    /* the revealed cell at (c_y, l_y) in both realisations, the rest refit */
    or_refit(p, p->prior, cell, cy, ly, cm, cp, tp, tm);
    int rc = solve(p, cm, tm, solver, minus);
    if (!rc) rc = solve(p, cp, tp, solver, plus);
    free(cm);
    *c_y = cy;
    *l_y = ly;
    return rc;
}

int or_score(const or_problem *p, const float *cap_lo, const float *cap_hi,
             const float *tail_lo, const float *tail_hi, const float *qn, int Q,
             uint64_t seed, uint32_t stream_id, uint32_t round,
             int n_cand, const int32_t *cand, int O, int S, int solver,
             int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed,
             float *gamma_t, int32_t *best, float *dump_t)
{
    if (n_cand < 0 || O < 1 || S < 1 || Q % O != 0) return -1;
    if ((int64_t)O * S > ((int64_t)1 << 22)) return -1;
    int cells = cells_of(p);
    for (int e = 0; e < n_cand; ++e)
        if (cand[e] < 0 || cand[e] >= cells) return -1;

    or_alloc am, ap;
    float gt;
    int rc = or_base_gap(p, cap_lo, cap_hi, tail_lo, tail_hi, solver, &am, &ap, &gt);
    if (rc) return rc;
    *gamma_t = gt;
    const int64_t g_t = llrintf(gt * 0x1p40f);
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
        int64_t tot = 0;
        for (int o = 0; o < O; ++o) {
            int64_t acc = 0;
            for (int s = 0; s < S; ++s) {
                int32_t kc, kl;
                or_draw_index(seed, stream_id, round, cell, Q, O, o, s, &kc, &kl);
                float cy = or_map(cap_lo[cell], cap_hi[cell], qn[kc]);
                float ly = or_map(tail_lo[cell], tail_hi[cell], qn[kl]);
                restore_row(p, cell, cap_lo, cap_hi, tail_lo, tail_hi, cm, cp, tp, tm);
                or_refit(p, p->prior, cell, cy, ly, cm, cp, tp, tm);
                rc = solve(p, cm, tm, solver, &am);
                if (!rc) rc = solve(p, cp, tp, solver, &ap);
                if (rc) { free(cm); return rc; }
                float g = ap.t_star - am.t_star;          /* Gamma_{t+1} of this scenario */
                acc += llrintf(g * 0x1p40f);
                if (dump_t) {
                    size_t idx = (((size_t)e * O + o) * S + s) * 2;
                    dump_t[idx] = am.t_star;
                    dump_t[idx + 1] = ap.t_star;
                }
            }
            if (sum_eo) sum_eo[(size_t)e * O + o] = acc;
            tot += acc;
        }
        restore_row(p, cell, cap_lo, cap_hi, tail_lo, tail_hi, cm, cp, tp, tm);

        int64_t sc = g_t * n - tot;                        /* sum of Gamma_t - Gamma_{t+1} */
        if (gap) gap[e] = ((double)tot * 0x1p-40) / (double)n;
        if (score) score[e] = ((double)sc * 0x1p-40) / (double)n;
        if (score_fixed) score_fixed[e] = sc;
        /* Largest expected reduction; ties: fewer profiling GPU-seconds
         * (300 s x TP, Section 4.3 and 5), then earlier position. */
        int j = (cell / p->B) % OR_T;
        if (best_e < 0 || sc > best_sc ||
            (sc == best_sc && j < (cand[best_e] / p->B) % OR_T)) {
            best_e = e;
            best_sc = sc;
        }
    }
    free(cm);
    if (best) *best = best_e >= 0 ? cand[best_e] : -1;
    return 0;
}

/*
 * Section 4.3, the last step: from the fixed-point sums of every
 * (candidate, outcome) pair, E[Gamma_{t+1} | e] = sum g 2^-40 / (O S), the
 * score E[Gamma_t - Gamma_{t+1} | e] and the argmax (largest score, then
 * fewer profiling GPU-seconds, i.e. lower TP, then earlier position). The
 * same rules as at the end of or_score, applied to sums computed elsewhere
 * (by or_score_cached over disjoint candidate ranges).
 */
int or_reduce(const or_problem *p, int n_cand, const int32_t *cand, int O, int S, float gamma_t,
              const int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed, int32_t *best)
{
    if (n_cand < 0 || O < 1 || S < 1) return -1;
    const int64_t g_t = llrintf(gamma_t * 0x1p40f);
    const int64_t n = (int64_t)O * S;
    int best_e = -1;
    int64_t best_sc = 0;
    for (int e = 0; e < n_cand; ++e) {
        int64_t tot = 0;
        for (int o = 0; o < O; ++o) tot += sum_eo[(size_t)e * O + o];
        int64_t sc = g_t * n - tot;
        if (gap) gap[e] = ((double)tot * 0x1p-40) / (double)n;
        if (score) score[e] = ((double)sc * 0x1p-40) / (double)n;
        if (score_fixed) score_fixed[e] = sc;
        int j = (cand[e] / p->B) % OR_T;
        if (best_e < 0 || sc > best_sc ||
            (sc == best_sc && j < (cand[best_e] / p->B) % OR_T)) {
            best_e = e;
            best_sc = sc;
        }
    }
    if (best) *best = best_e >= 0 ? cand[best_e] : -1;
    return 0;
}

/*
 * The fixed-point sums of or_score, scenario for scenario, with each
 * candidate's solves cached. Both solvers read a cell's tail only through
 * the SLO test tail <= L_i (Eq. 5), and c_y is a function of the capacity
 * position k_cap alone, so under the revealed-only prior a scenario's two
 * allocations, and its Gamma', depend on its draw only through the pair
 * (k_cap, l_y <= L_i); under the monotone prior l_y also moves the tail
 * bounds of the row's other bins, so the key is (k_cap, k_tail). A scenario
 * whose pair was met before in the same candidate reuses that scenario's
 * rint(Gamma' 2^40); every other step (draws, maps, patches, solves, sums)
 * is or_score's. Used to compute expected sums of workloads too large for
 * or_score; the tests hold the two equal wherever or_score finishes.
 * sum_eo [n_cand][O] is required; gamma_t receives Gamma_t.
 */
int or_score_cached(const or_problem *p, const float *cap_lo, const float *cap_hi,
                    const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                    uint64_t seed, uint32_t stream_id, uint32_t round,
                    int n_cand, const int32_t *cand, int O, int S, int solver,
                    int64_t *sum_eo, float *gamma_t)
{
    if (n_cand < 0 || O < 1 || S < 1 || Q < 1 || Q % O != 0 || !sum_eo) return -1;
    if ((int64_t)O * S > ((int64_t)1 << 22)) return -1;
    int cells = cells_of(p);
    for (int e = 0; e < n_cand; ++e)
        if (cand[e] < 0 || cand[e] >= cells) return -1;

    or_alloc am, ap;
    float gt;
    int rc = or_base_gap(p, cap_lo, cap_hi, tail_lo, tail_hi, solver, &am, &ap, &gt);
    if (rc) return rc;
    if (gamma_t) *gamma_t = gt;

    float *cm = (float *)malloc(sizeof(float) * cells * 4);
    /* key: (k_cap, gate) under the revealed-only prior, (k_cap, k_tail
     * within the stratum) under the monotone prior */
    const size_t nkey = p->prior == OR_PRIOR_REVEALED ? 2 * (size_t)Q : (size_t)Q * (size_t)(Q / O);
    int64_t *memo = (int64_t *)malloc(sizeof(int64_t) * nkey);
    uint8_t *known = (uint8_t *)malloc(nkey);
    if (!cm || !memo || !known) { free(cm); free(memo); free(known); return -2; }
    float *tm = cm + cells, *cp = cm + 2 * cells, *tp = cm + 3 * cells;
    memcpy(cm, cap_lo, sizeof(float) * cells);
    memcpy(tm, tail_hi, sizeof(float) * cells);
    memcpy(cp, cap_hi, sizeof(float) * cells);
    memcpy(tp, tail_lo, sizeof(float) * cells);

    for (int e = 0; e < n_cand; ++e) {
        const int32_t cell = cand[e];
        const float L = p->slo[cell / (OR_T * p->B)];
        memset(known, 0, nkey);
        for (int o = 0; o < O; ++o) {
            int64_t acc = 0;
            for (int s = 0; s < S; ++s) {
                int32_t kc, kl;
                or_draw_index(seed, stream_id, round, cell, Q, O, o, s, &kc, &kl);
                float cy = or_map(cap_lo[cell], cap_hi[cell], qn[kc]);
                float ly = or_map(tail_lo[cell], tail_hi[cell], qn[kl]);
                size_t key = p->prior == OR_PRIOR_REVEALED ? 2 * (size_t)kc + (ly <= L ? 1u : 0u)
                                                           : (size_t)kc * (size_t)(Q / O) + (size_t)(kl % (Q / O));
                if (!known[key]) {
                    restore_row(p, cell, cap_lo, cap_hi, tail_lo, tail_hi, cm, cp, tp, tm);
                    or_refit(p, p->prior, cell, cy, ly, cm, cp, tp, tm);
                    rc = solve(p, cm, tm, solver, &am);
                    if (!rc) rc = solve(p, cp, tp, solver, &ap);
                    if (rc) { free(cm); free(memo); free(known); return rc; }
                    float g = ap.t_star - am.t_star;
                    memo[key] = llrintf(g * 0x1p40f);
                    known[key] = 1;
                }
                acc += memo[key];
            }
            sum_eo[(size_t)e * O + o] = acc;
        }
        restore_row(p, cell, cap_lo, cap_hi, tail_lo, tail_hi, cm, cp, tp, tm);
    }
    free(cm); free(memo); free(known);
    return 0;
}

/*
 * Section 4.2: certified infeasible when even A+ cannot meet the critical
 * floors; certified feasible when A- meets them, the gap is at most eps and
 * every cell that A- commits replicas to has been measured (its tail upper
 * bound is known; A- already keeps it within the SLO); otherwise undecided.
 * Without critical classes both realisations meet the (empty) floors.
 */
int or_certificate(const or_problem *p, const float *cap_lo, const float *cap_hi,
                   const float *tail_lo, const float *tail_hi, const uint8_t *revealed,
                   float eps, int solver, int *state, float *gamma_t)
{
    or_alloc am, ap;
    float gt;
    int rc = or_base_gap(p, cap_lo, cap_hi, tail_lo, tail_hi, solver, &am, &ap, &gt);
    if (rc) return rc;
    int committed_known = 1;
    for (int i = 0; i < p->K; ++i) {
        if (am.replicas[i] <= 0) continue;
        int j = 0;
        while (j < OR_T && (1 << j) != am.tp[i]) ++j;
        int cell = (i * OR_T + j) * p->B + am.bin[i];
        if (!revealed[cell]) committed_known = 0;
    }
    *gamma_t = gt;
    if (!ap.floors_met) *state = 2;
    else *state = (am.floors_met && gt <= eps && committed_known) ? 1 : 0;
    return 0;
}

/*
 * Algorithm 1 on one reveal order: common initial design (the first r0
 * cells of perm), then per round: A-, A+, certificate; stop when it fires
 * (certified feasible or certified infeasible),
 * else reveal the candidate with the largest score (ties: lower TP, then
 * earlier in perm). Revealing sets lo = hi = the hidden true value. Each
 * revealed cell costs 300 s x TP GPU-seconds (Section 5). Trajectories are
 * parity unpinned against the paper (its measured grid is not available).
 * policy 1 replaces the scored choice by the next unrevealed cell of perm:
 * the fixed-order baselines of Section 6.2 (uniform random when perm is a
 * random permutation, fixed grid order when it lists the grid), stopped by
 * the same certificate.
 */
static int replay_impl(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                       const float *prior_tail_lo, const float *prior_tail_hi,
                       const float *truth_cap, const float *truth_tail, const int32_t *perm,
                       int r0, float eps, const float *qn, int Q, uint64_t seed,
                       uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                       int cached, int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                       double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                       float *gamma_trace);

int or_replay_stream(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                     const float *prior_tail_lo, const float *prior_tail_hi,
                     const float *truth_cap, const float *truth_tail, const int32_t *perm,
                     int r0, float eps, const float *qn, int Q, uint64_t seed,
                     uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                     int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                     double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                     float *gamma_trace)
{
    return replay_impl(p, prior_cap_lo, prior_cap_hi, prior_tail_lo, prior_tail_hi, truth_cap, truth_tail,
                       perm, r0, eps, qn, Q, seed, stream_id, O, S, max_rounds, solver, policy, 0, rounds,
                       reveal_order, n_revealed, gpu_seconds, state, final_minus, gamma_trace);
}

/* The same replay with each round's scores from or_score_cached + or_reduce
 * (the same sums and argmax, fewer solves); the tests hold the two equal. */
int or_replay_stream_cached(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                            const float *prior_tail_lo, const float *prior_tail_hi,
                            const float *truth_cap, const float *truth_tail, const int32_t *perm,
                            int r0, float eps, const float *qn, int Q, uint64_t seed,
                            uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                            int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                            double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                            float *gamma_trace)
{
    return replay_impl(p, prior_cap_lo, prior_cap_hi, prior_tail_lo, prior_tail_hi, truth_cap, truth_tail,
                       perm, r0, eps, qn, Q, seed, stream_id, O, S, max_rounds, solver, policy, 1, rounds,
                       reveal_order, n_revealed, gpu_seconds, state, final_minus, gamma_trace);
}

static int replay_impl(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                       const float *prior_tail_lo, const float *prior_tail_hi,
                       const float *truth_cap, const float *truth_tail, const int32_t *perm,
                       int r0, float eps, const float *qn, int Q, uint64_t seed,
                       uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                       int cached, int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                       double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                       float *gamma_trace)
{
    int cells = cells_of(p);
    if (r0 < 0 || r0 > cells || policy < 0 || policy > 1) return -1;
    float *buf = (float *)malloc(sizeof(float) * cells * 4);
    uint8_t *rev = (uint8_t *)calloc(cells, 1);
    int32_t *cand = (int32_t *)malloc(sizeof(int32_t) * cells);
    if (!buf || !rev || !cand) { free(buf); free(rev); free(cand); return -2; }
    float *clo = buf, *chi = buf + cells, *tlo = buf + 2 * cells, *thi = buf + 3 * cells;
    memcpy(clo, prior_cap_lo, sizeof(float) * cells);
    memcpy(chi, prior_cap_hi, sizeof(float) * cells);
    memcpy(tlo, prior_tail_lo, sizeof(float) * cells);
    memcpy(thi, prior_tail_hi, sizeof(float) * cells);
    int nrev = 0;
    double gs = 0.0;
    for (int q = 0; q < r0; ++q) {
        int c = perm[q];
        or_refit(p, p->prior, c, truth_cap[c], truth_tail[c], clo, chi, tlo, thi);
        rev[c] = 1;
        reveal_order[nrev++] = c;
        gs += 300.0 * (double)(1 << ((c / p->B) % OR_T));
    }
    int rc = 0, st = 0, r = 0;
    for (;;) {
        int z;
        float gt;
        rc = or_certificate(p, clo, chi, tlo, thi, rev, eps, solver, &z, &gt);
        if (rc) break;
        if (gamma_trace) gamma_trace[r] = gt;
        if (z != 0) { st = z; break; }
        int nc = 0;
        for (int q = 0; q < cells; ++q)
            if (!rev[perm[q]]) cand[nc++] = perm[q];
        if (nc == 0 || r >= max_rounds) { st = 0; break; }
        int32_t bestc = cand[0];
        if (policy == 0 && !cached) {
            float g2;
            rc = or_score(p, clo, chi, tlo, thi, qn, Q, seed, stream_id, (uint32_t)r, nc, cand, O, S,
                          solver, NULL, NULL, NULL, NULL, &g2, &bestc, NULL);
            if (rc) break;
        } else if (policy == 0) {
            float g2;
            int64_t *se = (int64_t *)malloc(sizeof(int64_t) * (size_t)nc * O);
            if (!se) { rc = -2; break; }
            rc = or_score_cached(p, clo, chi, tlo, thi, qn, Q, seed, stream_id, (uint32_t)r, nc, cand, O, S,
                                 solver, se, &g2);
            if (!rc) rc = or_reduce(p, nc, cand, O, S, g2, se, NULL, NULL, NULL, &bestc);
            free(se);
            if (rc) break;
        }
        or_refit(p, p->prior, bestc, truth_cap[bestc], truth_tail[bestc], clo, chi, tlo, thi);
        rev[bestc] = 1;
        reveal_order[nrev++] = bestc;
        gs += 300.0 * (double)(1 << ((bestc / p->B) % OR_T));
        ++r;
    }
    if (!rc) {
        or_alloc ap;
        float gt;
        rc = or_base_gap(p, clo, chi, tlo, thi, solver, final_minus, &ap, &gt);
    }
    *rounds = r;
    *n_revealed = nrev;
    *gpu_seconds = gs;
    *state = st;
    free(buf); free(rev); free(cand);
    return rc;
}
