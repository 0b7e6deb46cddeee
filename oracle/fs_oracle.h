/*
 * CPU oracle for the FleetSieve decision-gap computation.
 *
 * TEST INFRASTRUCTURE ONLY. Plain, slow, single-threaded C that states the
 * method as directly as possible so that the CUDA library can be checked
 * against it. Only the tests, the smoke check and the benchmark's CPU
 * baseline may load it; the product path never does. It shares no code,
 * header, table or constant generator with the CUDA library.
 *
 * Build with -O2 -ffp-contract=off -fno-fast-math: every float operation
 * below is one IEEE round-to-nearest operation, never a fused multiply-add.
 *
 * Sources (FleetSieve, "Decision-Critical Profiling for SLO-Aware LLM Fleet
 * Configuration"):
 *   Section 3, Eqs. 1-5 and the lexicographic objective: the allocation
 *     model (one homogeneous configuration per class, integer replicas,
 *     served load x_i <= n c, GPU budget G, tail gate l <= L_i, r_i = x/lambda);
 *     tier 1, the fulfilment floors delta_i of the critical classes;
 *   Section 4.1: conservative A- (lower capacity, upper tail) and optimistic
 *     A+ (upper capacity, lower tail) realisations;
 *   Section 4.2: the allocation gap and the certificate;
 *   Section 4.3: score_t(e) = E[Gamma_t - Gamma_{t+1} | e];
 *   Algorithm 1: the profiling loop;
 *   Section 5 (System): 300 s per cell, GPU-seconds = duration x TP.
 * The threshold solver (largest t whose cheapest per-class cover fits G)
 * fixes tier 2 of the objective where the paper leaves the algorithm open.
 *
 * Parity pins (tests/): brute-force enumeration, the paper's Table 2/3
 * allocation and the C128 tail rejection, Philox known-answer vectors,
 * closed-form quantile CDF, invariants. Pieces without such a pin say
 * "parity unpinned" where they are defined.
 */
#ifndef FS_ORACLE_H
#define FS_ORACLE_H

#include <stdint.h>

#define OR_T 4          /* TP degrees {1, 2, 4, 8} */
#define OR_KMAX 64      /* classes */

typedef struct {
    int K;              /* classes */
    int B;              /* load bins per (class, TP) */
    int G;              /* GPU budget, Eq. 3 */
    const float *demand;/* lambda_i [K], req/s */
    const float *slo;   /* L_i [K], seconds */
    const float *floor; /* delta_i [K] in [0, 1], tier 1 of Section 3; 0 = class i is
                           not critical; NULL = no critical class */
    int prior;          /* interval refit after a measurement (prior.c): OR_PRIOR_REVEALED
                           or OR_PRIOR_MONOTONE */
} or_problem;

#define OR_PRIOR_REVEALED 0  /* only the measured cell collapses */
#define OR_PRIOR_MONOTONE 1  /* and its row's other bins are refit (nondecreasing in load) */

/* One allocation. A class with replicas[i] == 0 has tp = 0, bin = -1. */
typedef struct {
    float t_star;               /* max-min fulfilment reached, 0 if none */
    int32_t total_gpus;         /* sum of n * tau */
    int32_t ok;                 /* t_star > 0 */
    int32_t floors_met;         /* every critical class can reach its floor within G */
    uint64_t has_option_mask;   /* bit i: class i has an SLO-feasible cell */
    int32_t tp[OR_KMAX];
    int32_t bin[OR_KMAX];
    int32_t replicas[OR_KMAX];
    float fulfil[OR_KMAX];
} or_alloc;

/* Sampler: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11). */
void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
/* Symmetric triangular quantile table on [0, 1], Q entries. */
void or_triangular_table(int Q, float *qn);
/* Quantile indices of one scenario (candidate cell, outcome o, sample s). */
int or_draw_index(uint64_t seed, uint32_t stream_id, uint32_t round, int32_t cell,
                  int Q, int O, int o, int s, int32_t *k_cap, int32_t *k_tail);
/* Affine map of a quantile value into [lo, hi]. */
float or_map(float lo, float hi, float q);

/* Fulfilment of n replicas of capacity c for demand lam. */
float or_fulfil(int n, float c, float lam);

/* Allocation solvers on one realisation (cap, tail are [K][4][B]). */
int or_solve_literal(const or_problem *p, const float *cap, const float *tail, or_alloc *out);
int or_solve_frontier(const or_problem *p, const float *cap, const float *tail, or_alloc *out);
/* Max-min fulfilment and goodput of a given allocation (tp index -1 = none). */
int or_evaluate(const or_problem *p, const float *cap, const float *tail,
                const int32_t *tp_index, const int32_t *bin, const int32_t *replicas,
                double *max_min, double *goodput);

/* Base solves A-, A+ and the gap Gamma_t = t*(A+) - t*(A-). */
int or_base_gap(const or_problem *p, const float *cap_lo, const float *cap_hi,
                const float *tail_lo, const float *tail_hi, int solver,
                or_alloc *minus, or_alloc *plus, float *gamma_t);

/* One scenario: draw, patch both realisations, solve both. */
int or_scenario(const or_problem *p, const float *cap_lo, const float *cap_hi,
                const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                uint64_t seed, uint32_t stream_id, uint32_t round, int32_t cell,
                int O, int o, int s, int solver,
                float *c_y, float *l_y, or_alloc *minus, or_alloc *plus);

/* Monte-Carlo score of every candidate (Section 4.3). */
int or_score(const or_problem *p, const float *cap_lo, const float *cap_hi,
             const float *tail_lo, const float *tail_hi, const float *qn, int Q,
             uint64_t seed, uint32_t stream_id, uint32_t round,
             int n_cand, const int32_t *cand, int O, int S, int solver,
             int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed,
             float *gamma_t, int32_t *best, float *dump_t /* [n_cand*O*S*2] or NULL */);

/* The same fixed-point sums with each candidate's solves cached by
 * (capacity position, tail within SLO); Gamma_t into gamma_t (nullable). */
int or_score_cached(const or_problem *p, const float *cap_lo, const float *cap_hi,
                    const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                    uint64_t seed, uint32_t stream_id, uint32_t round,
                    int n_cand, const int32_t *cand, int O, int S, int solver,
                    int64_t *sum_eo /* [n_cand*O] */, float *gamma_t);

/* Expectations, scores and argmax (Section 4.3) from the sums. */
int or_reduce(const or_problem *p, int n_cand, const int32_t *cand, int O, int S, float gamma_t,
              const int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed, int32_t *best);

/* Collapse cell to the measurement (c, l) and refit the other intervals under
 * the given prior (Section 4.1; prior.c), in place. */
int or_refit(const or_problem *p, int prior, int32_t cell, float c, float l,
             float *cap_lo, float *cap_hi, float *tail_lo, float *tail_hi);

/* Tiers 3-4 of the lexicographic objective (lexicographic.c): the allocation
 * keeping tiers 1-2 optimal with the most goodput, then the fewest GPUs, then
 * the tie rules class by class; *goodput_fx = its goodput in 2^-20 req/s. */
int64_t or_goodput_fx(int n, float c, float lam);
int or_solve_lex(const or_problem *p, const float *cap, const float *tail, int solver,
                 or_alloc *out, int64_t *goodput_fx);
/* A-, A+ to tier 4; the max-min gap and the goodput gap |GP+ - GP-| / sum lambda. */
int or_base_gap_lex(const or_problem *p, const float *cap_lo, const float *cap_hi,
                    const float *tail_lo, const float *tail_hi, int solver,
                    or_alloc *minus, or_alloc *plus, int64_t *gp_minus, int64_t *gp_plus,
                    float *gamma_mm, double *gamma_gp);
/* Stage-wise certificate: both gaps at most eps. */
int or_certificate_lex(const or_problem *p, const float *cap_lo, const float *cap_hi,
                       const float *tail_lo, const float *tail_hi, const uint8_t *revealed,
                       float eps, int solver, int *state, float *gamma_mm, double *gamma_gp);
/* The goodput stage of the Monte-Carlo score (sums in 2^-20 req/s). */
int or_score_goodput(const or_problem *p, const float *cap_lo, const float *cap_hi,
                     const float *tail_lo, const float *tail_hi, const float *qn, int Q,
                     uint64_t seed, uint32_t stream_id, uint32_t round,
                     int n_cand, const int32_t *cand, int O, int S, int solver,
                     int64_t *sum_eo, double *gap, double *score, int64_t *score_fixed,
                     int64_t *gamma_fx, double *gamma_gp, int32_t *best);

/* Certificate (Section 4.2): 0 undecided, 1 certified feasible, 2 certified
 * infeasible (even A+ misses a critical floor). */
int or_certificate(const or_problem *p, const float *cap_lo, const float *cap_hi,
                   const float *tail_lo, const float *tail_hi, const uint8_t *revealed,
                   float eps, int solver, int *state, float *gamma_t);

/* Algorithm 1 on one reveal order; policy 0 reveals the best-scored cell,
 * policy 1 the next unrevealed cell of perm (the fixed-order baselines). */
int or_replay_stream(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                     const float *prior_tail_lo, const float *prior_tail_hi,
                     const float *truth_cap, const float *truth_tail, const int32_t *perm,
                     int r0, float eps, const float *qn, int Q, uint64_t seed,
                     uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                     int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                     double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                     float *gamma_trace);

/* The same replay with each round scored by or_score_cached + or_reduce. */
int or_replay_stream_cached(const or_problem *p, const float *prior_cap_lo, const float *prior_cap_hi,
                            const float *prior_tail_lo, const float *prior_tail_hi,
                            const float *truth_cap, const float *truth_tail, const int32_t *perm,
                            int r0, float eps, const float *qn, int Q, uint64_t seed,
                            uint32_t stream_id, int O, int S, int max_rounds, int solver, int policy,
                            int32_t *rounds, int32_t *reveal_order, int32_t *n_revealed,
                            double *gpu_seconds, int32_t *state, or_alloc *final_minus,
                            float *gamma_trace);

#endif
