/*
 * Oracle interval refit after a measurement (Section 4.1, Algorithm 1's
 * "fit joint capacity and tail intervals").
 *
 * TEST INFRASTRUCTURE ONLY (see fs_oracle.h).
 *
 * The paper keeps per-cell capacity and tail intervals that "combine an
 * interior-knee structural prior with measured residuals", without giving
 * the prior's form, and names a revealed-only variant. Two priors:
 *
 *   OR_PRIOR_REVEALED (0): a measurement collapses its own cell's intervals
 *     to the measured values; no other cell changes.
 *   OR_PRIOR_MONOTONE (1): the reading of the interior-knee prior. Within
 *     one (class, TP) row the load bins are ordered by offered load, and
 *     both the sustainable throughput and the binding tail latency are
 *     nondecreasing in the load bin (throughput rises with offered load and
 *     the tail grows with it, so the SLO-feasible peak is an interior knee
 *     where the tail meets the SLO). A measurement (c, l) of bin b_e then
 *     bounds the row's other bins: for b > b_e, c_b >= c and l_b >= l; for
 *     b < b_e, c_b <= c and l_b <= l. Each interval is intersected with
 *     that half-line, clamped so that it never empties: a lower bound rises
 *     to min(max(lo, v), hi), an upper bound falls to max(min(hi, v), lo).
 *     Cells of other rows keep their intervals.
 *
 * Properties the tests hold it to: no interval ever widens; the measured
 * cell holds exactly its values; other rows are unchanged; a truth table
 * that is monotone in the load bin and lies inside the intervals still lies
 * inside them after any sequence of refits by its own values. The form of
 * the paper's prior (and its residual bands) is not given: parity unpinned
 * against the paper beyond these properties.
 */
#include "fs_oracle.h"

static float raise_lo(float lo, float hi, float v)
{
    float x = lo > v ? lo : v;      /* max(lo, v) */
    return x < hi ? x : hi;         /* then at most hi */
}

static float lower_hi(float lo, float hi, float v)
{
    float x = hi < v ? hi : v;      /* min(hi, v) */
    return x > lo ? x : lo;         /* then at least lo */
}

int or_refit(const or_problem *p, int prior, int32_t cell, float c, float l,
             float *cap_lo, float *cap_hi, float *tail_lo, float *tail_hi)
{
    int cells = p->K * OR_T * p->B;
    if (cell < 0 || cell >= cells || prior < 0 || prior > 1) return -1;
    cap_lo[cell] = cap_hi[cell] = c;
    tail_lo[cell] = tail_hi[cell] = l;
    if (prior == OR_PRIOR_REVEALED) return 0;
    int row = cell / p->B, be = cell % p->B;
    for (int b = 0; b < p->B; ++b) {
        int x = row * p->B + b;
        if (b > be) {           /* higher load: at least the measured values */
            cap_lo[x] = raise_lo(cap_lo[x], cap_hi[x], c);
            tail_lo[x] = raise_lo(tail_lo[x], tail_hi[x], l);
        } else if (b < be) {    /* lower load: at most the measured values */
            cap_hi[x] = lower_hi(cap_lo[x], cap_hi[x], c);
            tail_hi[x] = lower_hi(tail_lo[x], tail_hi[x], l);
        }
    }
    return 0;
}
