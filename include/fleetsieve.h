/*
 * fleetsieve.h -- C ABI of the GB300 decision-gap scorer.
 *
 * FleetSieve (decision-critical profiling for SLO-aware LLM fleet
 * configuration) chooses which serving configuration to measure next by the
 * expected reduction of the gap between a conservative and an optimistic
 * fleet allocation. This library evaluates that expectation by Monte Carlo
 * on one GPU (sm_103a):
 *
 *   fs_load_model         bounds, SLOs, demands, G  -> device-resident model
 *   fs_score_candidates   samples                   -> E[Gamma_{t+1} | e], score, argmax
 *   fs_solve(_batch)      realisation               -> allocation
 *   fs_solve_bounds       conservative / optimistic allocations and Gamma_t
 *   fs_set_floors         critical classes' fulfilment floors (tier 1)
 *   fs_reveal, fs_certificate, fs_replay            the profiling loop
 *
 * Notation (paper, Section 3): class i has demand lambda_i (req/s) and an SLO
 * L_i (s) on its binding tail metric. A configuration is a TP degree
 * tau in {1, 2, 4, 8} (index j = 0..3) and a load bin b; a replica of it uses
 * tau GPUs and serves c req/s with tail l. Cells are indexed
 * cell = (i * 4 + j) * B + b and every per-cell array is [K][4][B] row-major.
 *
 * Conventions for every call:
 *   - returns FS_OK (0) or a negative FS_E* code; fs_last_error() gives a
 *     thread-local message for the last failure of the calling thread;
 *   - no exception or abort crosses the ABI;
 *   - the caller owns every buffer it passes; inputs are copied (host inputs
 *     before the call returns, device inputs in stream order);
 *   - calls taking host output pointers are synchronous; calls named
 *     *_async / *_batch take device pointers and a cudaStream_t (as void*),
 *     enqueue their work and return; fs_check() synchronises such a stream and
 *     reports device-side errors;
 *   - one fs_model is not thread-safe; separate models are independent.
 */
#ifndef FLEETSIEVE_H
#define FLEETSIEVE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    FS_OK = 0,
    FS_EINVAL = -1,   /* bad argument: NaN/inf, lo > hi, sizes out of range, ... */
    FS_ENOMEM = -2,   /* device or host allocation failed */
    FS_ECUDA = -3,    /* a CUDA runtime call failed */
    FS_ETIMEOUT = -4, /* a bounded device wait ran out (watchdog) */
    FS_EDEVICE = -5   /* a kernel reported an inconsistency in its status word */
};

#define FS_TP_COUNT 4        /* TP degrees {1, 2, 4, 8} */
#define FS_MAX_CLASSES 64    /* K */
#define FS_MAX_BINS 4096     /* B */
#define FS_MAX_GPUS 32767    /* G */
#define FS_MAX_THRESHOLDS 16384 /* K * sum_tau floor(G / tau) must not exceed this */
#define FS_MAX_SAMPLES_PER_CAND (1 << 22) /* O * S */

typedef struct fs_model fs_model;

/*
 * Per-cell uncertainty state after round t (Section 4.1): capacity interval
 * [cap_lo, cap_hi] (req/s per replica) and tail interval [tail_lo, tail_hi]
 * (s). All four arrays are host pointers to [K][4][B] floats, finite, >= 0,
 * lo <= hi. revealed: optional host [K][4][B] flags (nonzero = the cell was
 * measured, Algorithm 1's "reveal"; its bounds must then be collapsed,
 * lo == hi, else FS_EINVAL); NULL = no cell measured yet. The certificate
 * (Section 4.2) reads these flags. quantile: optional host table Qn[Q] in
 * [0, 1], nondecreasing, of the posterior inside an interval (value
 * v = lo + (hi - lo) * Qn[k]); NULL selects the built-in symmetric
 * triangular table with Q = 4096. Q must be a power of two >= 4.
 */
typedef struct {
    int32_t K;
    int32_t B;
    const float *cap_lo;
    const float *cap_hi;
    const float *tail_lo;
    const float *tail_hi;
    const uint8_t *revealed;
    const float *quantile;
    int32_t Q;
    int32_t reserved;
} fs_bounds;

/*
 * fs_load_model -- upload bounds, SLOs L_i (s, > 0), demands lambda_i
 * (req/s, > 0) and the GPU budget G (Section 3, Eqs. 1-5) into a new model.
 * cuda_stream: stream used by the synchronous calls of this model (NULL =
 * default stream). Limits: 1 <= K <= 64, 1 <= B <= 4096, 1 <= G <= 32767,
 * K * (floor(G/1) + floor(G/2) + floor(G/4) + floor(G/8)) <= 16384.
 * Cells start revealed as bounds->revealed says (none when it is NULL), so a
 * model saved with fs_get_state resumes where it stopped (the counter-based
 * draws depend only on seed, stream, round and cell). *out is set only on
 * success.
 */
int fs_load_model(const fs_bounds *bounds, const float *slo, const float *demand, int32_t G,
                  void *cuda_stream, fs_model **out);

/*
 * fs_update_bounds -- replace the four bound arrays (host, [K][4][B]) of a
 * model, e.g. after the intervals were refit (Algorithm 1, "fit joint
 * capacity and tail intervals"). Revealed flags are kept. The arrays are
 * copied (into page-locked staging) before the call returns, which queues no
 * device work: the next call that needs the bounds on the device queues their
 * copy on the model's stream (work it queues on another stream waits for it),
 * and fs_score_candidates reads freshly staged bounds where they are. Every
 * later call on the model sees the new bounds.
 */
int fs_update_bounds(fs_model *m, const float *cap_lo, const float *cap_hi,
                     const float *tail_lo, const float *tail_hi);

/*
 * fs_set_floors -- fulfilment floors of the critical classes (Section 3,
 * tier 1 of the lexicographic objective: enforce r_i >= delta_i for critical
 * classes whenever feasible). floor: host [K] floats delta_i in [0, 1];
 * delta_i = 0 marks class i as not critical; NULL clears every floor (the
 * state a new model starts in). Under floors, every solve of this model
 * (fs_solve*, the scoring calls' realisations and scenarios, the
 * certificate, fs_replay) takes a critical class's options below its floor
 * as no options at all and maximises tier 2 over what remains; see
 * fs_allocation for the floor-only allocation. The values are copied before
 * the call returns and are in place for every later call on any stream.
 */
int fs_set_floors(fs_model *m, const float *floor);

/*
 * Monte-Carlo plan of one scoring call (Section 4.3).
 *   cand[n_cand]: candidate cell ids (host pointer for fs_score_candidates,
 *     device pointer for fs_score_candidates_async); duplicates allowed;
 *     revealed cells are allowed and score 0.
 *   O: outcome strata, a power of two dividing Q with Q/O <= 16384; S >= 1
 *     samples per (candidate, outcome); O * S <= 2^22.
 *   Draws: Philox4x32-10 (Salmon et al., SC'11) with key (seed_lo,
 *     seed_hi XOR stream_id) and counter (s/4, o, cell, round); sample s uses
 *     output word s mod 4, whose upper 16 bits give the capacity and lower 16
 *     bits the tail: the top log2(Q/O) bits of each half pick a quantile inside
 *     stratum o.
 */
typedef struct {
    uint64_t seed;
    uint32_t stream_id;
    uint32_t round;
    int32_t n_cand;
    int32_t O;
    int32_t S;
    int32_t reserved;
    const int32_t *cand;
} fs_samples;

/*
 * Per-scenario parity record written by the dump mode, one per scenario in
 * (candidate, outcome, sample) order, record stride fs_dump_stride(m) bytes:
 *   float c_y, l_y;          drawn capacity and tail of the candidate cell
 *   float t_star[2];         t* of the patched conservative [0] / optimistic [1] realisation
 *   int32_t total_gpus[2];
 *   uint32_t choice[2][K];   per class: replicas n (bits 0-15), TP index j
 *                            (bits 16-17), bin (bits 18-30); 0 = no replicas
 */
typedef struct {
    float c_y;
    float l_y;
    float t_star[2];
    int32_t total_gpus[2];
} fs_scenario_head;

/* Record stride of the dump for this model (bytes, a multiple of 8). */
int32_t fs_dump_stride(const fs_model *m);

/*
 * fs_score_candidates -- score_t(e) = E[Gamma_t - Gamma_{t+1} | e] for every
 * candidate (Section 4.3) with Gamma = t*(A+) - t*(A-) (Section 4.2, the
 * max-min gap). For every candidate e, outcome o and sample s the drawn
 * (c_y, l_y) replaces cell e in both the conservative (cap_lo, tail_hi) and
 * the optimistic (cap_hi, tail_lo) realisation, both allocations are solved,
 * and the gaps are summed in int64 fixed point (g = rint(Gamma' * 2^40)).
 * Host outputs (each nullable):
 *   gap_out[n_cand]   E[Gamma_{t+1} | e] = (sum g * 2^-40) / (O S)
 *   score_out[n_cand] (rint(Gamma_t 2^40) O S - sum g) * 2^-40 / (O S)
 *   gamma_t[1]        Gamma_t
 *   best[1]           argmax cell: largest score, then lower TP (fewer
 *                     profiling GPU-seconds, 300 s x TP), then earlier in cand;
 *                     -1 if n_cand == 0
 *   sum_eo[n_cand*O]  the int64 fixed-point sums per (candidate, outcome)
 * dump_dev: optional DEVICE buffer of n_cand*O*S*fs_dump_stride(m) bytes.
 */
int fs_score_candidates(fs_model *m, const fs_samples *samples, double *gap_out,
                        double *score_out, float *gamma_t, int32_t *best, int64_t *sum_eo,
                        void *dump_dev);

/* Same with samples->cand and every output on the device, enqueued on cuda_stream. */
int fs_score_candidates_async(fs_model *m, const fs_samples *samples, double *gap_dev,
                              double *score_dev, float *gamma_t_dev, int32_t *best_dev,
                              int64_t *sum_eo_dev, void *dump_dev, void *cuda_stream);

/*
 * fs_score_candidates_noalloc -- the same scores as fs_score_candidates, for
 * callers that cannot allocate device memory while they run: processes whose
 * device memory is already handed out by their own pool, and latency-critical
 * paths that must not pay for cudaMalloc/cudaFree (which can synchronise the
 * device). The paper has no counterpart; this entry point exists for them.
 * It allocates nothing and needs no fs_model:
 *   bounds_dev   DEVICE [4][K][4][B] floats: cap_lo, cap_hi, tail_lo, tail_hi
 *   slo_dev, demand_dev  DEVICE [K] floats
 *   quantile_dev DEVICE [Q] table, or NULL for the built-in triangular table
 *                (Q = 4096, rebuilt by every call)
 *   samples      as for fs_score_candidates_async (cand is a DEVICE pointer)
 *   gap_dev, score_dev [n_cand] doubles, gamma_t_dev [1], best_dev [1]: DEVICE
 *                outputs (each nullable)
 * The same limits as fs_load_model apply, and the values must satisfy its
 * rules (finite, >= 0 (-0.0 counts as 0), lo <= hi, SLOs and demands > 0):
 * they are on the device and are not checked here; candidate ids are
 * range-checked by the kernels (FS_EDEVICE). The kernels are the ones
 * fs_score_candidates runs, row tables included.
 * Scratch: all intermediates live in one fixed device array of 16 MiB
 * (16,777,216 bytes) that every GPU loading this library holds until the
 * process exits. A call takes the following pieces of it, each rounded up to
 * a multiple of 256 bytes, and returns FS_EINVAL without running when their
 * sum exceeds 16 MiB:
 *   4, 32 and 1024 bytes (status word, counters, reduction scratch);
 *   4 Q (only with quantile_dev NULL: the built-in table);
 *   8 T and 8, with T = K (floor(G/1) + floor(G/2) + floor(G/4) + floor(G/8))
 *     (thresholds and their counts);
 *   32 K twice (best capacity and bin per (class, TP) row), 1216 (the two
 *     base allocations), 65536 (their row tables);
 *   4 n I with n = max(n_cand, 1), I = 2 (20 + 3 P) + O (4 + 4 ceil(W / 4)),
 *     P the smallest power of two >= max(T + 1, 4), W = Q / O (the
 *     candidates' threshold tables and mapped quantile windows);
 *   8 n O (the fixed-point sums).
 * On the paper-scale grid (K = 2, G = 16, O = 8, Q = 4096) that allows 913
 * candidates per call.
 * Every call shares the array, which keeps the last call's contents (the
 * kernels clear what must start at zero): calls whose GPU work overlaps
 * (other streams or host threads) race. The call enqueues its kernels on
 * cuda_stream, copies the status word to the host and synchronises the
 * stream before it returns, reporting device-side errors (FS_ETIMEOUT,
 * FS_EDEVICE); it therefore cannot be captured into a CUDA graph.
 */
int fs_score_candidates_noalloc(int32_t K, int32_t B, int32_t G, const float *bounds_dev,
                                const float *slo_dev, const float *demand_dev,
                                const float *quantile_dev, int32_t Q, const fs_samples *samples,
                                double *gap_dev, double *score_dev, float *gamma_t_dev,
                                int32_t *best_dev, void *cuda_stream);

/*
 * One allocation (Section 3): per class the chosen TP degree (0 = none),
 * bin (-1 = none), replica count and fulfilment r_i; t_star = min_i r_i
 * reached (the tier-2 objective), ok = t_star > 0. floors_met = 1 when every
 * critical class can be served at its floor within G (always 1 without
 * floors). With ok = 0 and floors_met = 1 the critical classes still get
 * their cheapest options at or above their floors (same tie rules) and the
 * other classes nothing; with floors_met = 0 no class gets replicas.
 */
typedef struct {
    float t_star;
    int32_t total_gpus;
    uint64_t has_option_mask; /* bit i: class i has an SLO-feasible cell */
    int32_t ok;
    int32_t floors_met;
    int8_t tp[FS_MAX_CLASSES];
    int16_t bin[FS_MAX_CLASSES];
    int16_t replicas[FS_MAX_CLASSES];
    float fulfil[FS_MAX_CLASSES];
    double goodput;           /* served req/s sum_i min(lambda_i, n c) in steps of 2^-20
                                 (tier 3); filled under the lexicographic objective, else 0 */
} fs_allocation;

/*
 * fs_solve -- allocation of one realisation (host arrays cap, tail
 * [K][4][B]) under the model's SLOs, demands, floors and G. Tier 2 of the
 * objective (Section 3): t* is the largest option fulfilment t for which
 * every class's cheapest SLO-feasible option with fulfilment >= max(t,
 * delta_i) fits in G together; ties: lower TP, then fewer replicas, then
 * larger capacity, then lower bin; nothing fits -> t* = 0 and only the
 * floor-only allocation described at fs_allocation.
 */
int fs_solve(fs_model *m, const float *cap, const float *tail, fs_allocation *out);

/*
 * fs_solve_batch -- the allocation of Section 3 (Eqs. 1-5, the same solver
 * and tie rules as fs_solve) for n realisations at once: device arrays
 * cap_dev/tail_dev [n][K][4][B] (one realisation after another), out_dev [n]
 * device allocations. Enqueued on cuda_stream; inputs are read and outputs
 * written in stream order (the caller keeps them alive until then).
 */
int fs_solve_batch(fs_model *m, int32_t n, const float *cap_dev, const float *tail_dev,
                   fs_allocation *out_dev, void *cuda_stream);

/* A- and A+ at the current bounds (Section 4.1) and Gamma_t (host outputs, nullable). */
int fs_solve_bounds(fs_model *m, fs_allocation *minus, fs_allocation *plus, float *gamma_t);

/*
 * fs_reveal -- Algorithm 1's reveal step: cell has been measured (capacity
 * cap req/s per replica, binding tail tail s, both finite and >= 0). Its
 * intervals collapse to the measured values in both realisations
 * (Section 4.1: lo = hi), and it is marked revealed, which the certificate's
 * "committed tail upper bounds known" test reads (Section 4.2). Other cells
 * keep their intervals. Staged for the device like fs_update_bounds.
 */
int fs_reveal(fs_model *m, int32_t cell, float cap, float tail);

/*
 * fs_set_prior -- how a measurement updates the uncertainty state (Section
 * 4.1: intervals from an interior-knee structural prior plus measured
 * residuals; Algorithm 1 refits them after every reveal).
 *   FS_PRIOR_REVEALED (0, the state a new model starts in): the measured
 *     cell collapses to its values; no other cell changes (the revealed-only
 *     prior).
 *   FS_PRIOR_MONOTONE (1): the reading of the interior-knee prior used here:
 *     within a (class, TP) row, capacity and binding tail are nondecreasing
 *     in the load bin, so a measurement (c, l) of bin b also refits the row's
 *     other bins: for bins above b, lo = min(max(lo, v), hi); for bins below
 *     b, hi = max(min(hi, v), lo) (v = c for capacity, l for the tail); no
 *     interval ever widens or empties, and other rows do not change.
 * The prior applies to fs_reveal, to fs_replay's reveals and to every
 * scoring scenario (the drawn outcome refits the candidate's row in both
 * realisations before they are solved).
 */
#define FS_PRIOR_REVEALED 0
#define FS_PRIOR_MONOTONE 1
int fs_set_prior(fs_model *m, int32_t prior);

/*
 * fs_set_objective -- which tiers of Section 3's lexicographic objective the
 * solves of this model optimise.
 *   FS_OBJECTIVE_MAXMIN (0, the state a new model starts in): tiers 1-2
 *     (floors, then max min_i r_i by the threshold rule); the allocation is
 *     each class's cheapest cover at t*; fs_allocation.goodput is 0.
 *   FS_OBJECTIVE_LEXICOGRAPHIC (1): all four tiers. Among the allocations
 *     that keep tiers 1-2 optimal (every class at r_i >= max(t*, delta_i) when
 *     t* > 0; at t* = 0 the critical classes at their floors and the others
 *     free; nothing when the floors cannot be met): (3) the most served
 *     goodput sum_i min(lambda_i, n c), each class's term rounded to 2^-20
 *     req/s; (4) "minimise fragmentation" read as the fewest GPUs in use,
 *     then class by class the tie rules (no replicas, lower TP, fewer
 *     replicas, larger capacity, lower bin). fs_solve, fs_solve_batch and
 *     fs_solve_bounds return that allocation with its goodput, and
 *     fs_certificate becomes stage-wise (Section 4.2): certified feasible
 *     also needs the goodput gap |GP(A+) - GP(A-)| / sum_i lambda_i <= eps.
 *     Needs (K + 1)(G + 1) <= 4 Mi (FS_EINVAL otherwise). The scoring calls
 *     and fs_replay stay on the max-min stage; fs_score_goodput scores the
 *     goodput stage.
 */
#define FS_OBJECTIVE_MAXMIN 0
#define FS_OBJECTIVE_LEXICOGRAPHIC 1
int fs_set_objective(fs_model *m, int32_t objective);

/*
 * fs_score_goodput -- the goodput stage of Section 4.3's score (the second
 * curve of Fig. 4a): for every candidate e, outcome o and sample s the same
 * draw and realisations as fs_score_candidates (the model's prior and floors
 * included), both solved to tier 4, and the scenario's goodput gap
 * |GP(A+') - GP(A-')| summed in int64 units of 2^-20 req/s. Host outputs
 * (each nullable):
 *   gap_out[n_cand]   E[Gamma_gp,t+1 | e] = sum 2^-20 / (O S) / sum_i lambda_i
 *   score_out[n_cand] (Gamma_gp,t O S - sum) 2^-20 / (O S) / sum_i lambda_i
 *                     (Gamma_gp,t = |GP(A+) - GP(A-)| at the bounds, 2^-20 req/s)
 *   gamma_gp[1]       Gamma_gp,t / sum_i lambda_i
 *   best[1]           argmax: largest score, then lower TP, then earlier in cand
 *   sum_eo[n_cand*O]  the int64 sums
 * Needs sum_i lambda_i <= 2^20 req/s, G <= 1024, (K + 1)(G + 1) <= 4 Mi and
 * Q / O <= 4096 (2048 under the monotone prior: a segment's table of
 * positions lives in shared memory) (FS_EINVAL otherwise). Synchronous.
 * Independent of fs_set_objective.
 */
int fs_score_goodput(fs_model *m, const fs_samples *samples, double *gap_out, double *score_out,
                     double *gamma_gp, int32_t *best, int64_t *sum_eo);

/*
 * fs_get_state -- the model's current uncertainty state, for checkpointing
 * the profiling loop: bounds [K][4][B] (as staged by the last fs_load_model,
 * fs_update_bounds or fs_reveal) and revealed flags [K][4][B] (0 / 1) into
 * host arrays (each nullable). Loading them back through fs_bounds, with the
 * same SLOs, demands, G, quantile table and floors, gives a model whose every
 * later call returns what this one would.
 */
int fs_get_state(const fs_model *m, float *cap_lo, float *cap_hi, float *tail_lo, float *tail_hi,
                 uint8_t *revealed);

/*
 * Decision certificate (Section 4.2): *state = 2 (certified infeasible) when
 * even A+ misses a critical floor; 1 (certified feasible) when A- meets the
 * floors, Gamma_t <= eps and every cell to which A- commits replicas is
 * revealed; else 0 (undecided). Without floors state 2 cannot occur.
 * gamma_t nullable.
 */
int fs_certificate(fs_model *m, float eps, int32_t *state, float *gamma_t);

/*
 * fs_replay -- Algorithm 1 on n_streams independent reveal orders over the
 * model's bounds, batched on the device. Stream k: hidden truth
 * truth_cap/truth_tail[k][cells], order perm[k][cells] (its first r0 cells
 * are the common initial design; perm position breaks exact score ties).
 * Each round: A-, A+, certificate (eps, the model's floors); if undecided, score the unrevealed
 * cells (perm order) with O x S samples, Philox stream id k and round r,
 * then reveal the argmax. Stops on the certificate, when no cell is left, or
 * after max_rounds. policy 1 replaces the scored choice by the next
 * unrevealed cell of perm[k] (no scoring): the fixed-order baselines of
 * Section 6.2 (uniform random for a random perm, fixed grid order for a perm
 * that lists the grid), stopped by the same certificate. All inputs are host pointers; outputs host, nullable:
 *   rounds[k], state[k] (the certificate's 1 or 2, or 0 when the stream ran out
 *   of cells or rounds undecided), gpu_seconds[k] (300 s x TP per revealed cell),
 *   reveal_order[k][cells] (-1 padded), gamma_trace[k][max_rounds+1],
 *   final_minus[k] (A- at the end).
 */
typedef struct {
    int32_t n_streams;
    int32_t r0;
    float eps;
    int32_t O;
    int32_t S;
    int32_t max_rounds;
    int32_t policy;           /* 0: reveal the best-scored cell; 1: the next cell of perm */
    uint64_t seed;
    const float *truth_cap;
    const float *truth_tail;
    const int32_t *perm;
} fs_replay_spec;

int fs_replay(fs_model *m, const fs_replay_spec *spec, int32_t *rounds, int32_t *state,
              double *gpu_seconds, int32_t *reveal_order, float *gamma_trace,
              fs_allocation *final_minus);

/* Synchronise cuda_stream (NULL = the model's) and report device-side errors. */
int fs_check(fs_model *m, void *cuda_stream);

/*
 * Kernel timing for measurement (not part of the method). mode 1: every
 * later scoring call of this model records CUDA events around its
 * Monte-Carlo kernel on the stream it launches on; mode 2: also around the
 * base solves, the table preparation and the reduction; 0: off (up to 4096
 * calls are kept). fs_timing_enable also zeroes the model's work counts.
 * fs_timing_read waits for the recorded events and returns the summed
 * Monte-Carlo kernel time (ms), the number of timed calls, in mode 2
 * phase_ms[4] = summed (solve, prep, Monte-Carlo, reduction) time, and
 * work_counts[2] = what the Monte-Carlo kernel's table path did since the
 * counts were last zeroed: the t* its gap-table builds evaluated (at most two
 * per entry, once per segment; an entry whose capacity is at or below a
 * realisation's Cexcl takes that realisation's closed-gate t* without
 * evaluating it) and the scenarios that tested their tail gate (those of
 * strata whose tails lie on both sides of the SLO) (each output nullable); it
 * clears the record and the counts. Events between kernels also stop the
 * next kernel from starting early, so timed calls can take a little longer.
 */
int fs_timing_enable(fs_model *m, int32_t mode);
int fs_timing_read(fs_model *m, double *kernel_ms, int32_t *launches, double *phase_ms,
                   uint64_t *work_counts);

/*
 * Measurement floor (not part of the method). Times what the table path's
 * draws cost without the rest of the scorer, on the current device, over one
 * wave of 128-thread blocks (the table path's shape on large launches): each
 * block one segment, each thread an equal share of Philox4x32-10 calls
 * (counters as the scorer's), at least `calls` calls in all. mode 0: the
 * draws alone. mode 1: the draws with the table path's per-sample work
 * (capacity position from the word's top w bits, entry address, shared-memory
 * load, 64-bit sum) over a table of 2^w + 1 entries, with no chunks, staging,
 * table builds or barriers. Synchronous; allocates and frees its output
 * buffer. *ms = median of `reps` launches after three untimed ones;
 * *calls_done = the calls one launch made (>= calls). FS_EINVAL for a mode
 * other than 0/1, w outside [0, 12], calls outside [1, 2^36], reps outside
 * [1, 1000] or a null output.
 */
int fs_draw_floor(int32_t mode, int32_t w, int64_t calls, int32_t reps, double *ms, int64_t *calls_done);

/* Kernels this library has launched since it was loaded (all models). */
uint64_t fs_launch_count(void);

/*
 * Watchdog self-test: one kernel waits on a shared-memory barrier that no
 * copy ever completes, gives up after timeout_ns (clamped to [1 ms, 5 s]),
 * records the timeout in a status word and returns; the call then returns
 * FS_ETIMEOUT. Nothing is left running and the context stays usable.
 */
int fs_watchdog_selftest(int64_t timeout_ns);

void fs_free_model(fs_model *m);

const char *fs_last_error(void);

#ifdef __cplusplus
}
#endif

#endif
