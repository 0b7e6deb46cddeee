/*
 * Oracle sampler: counter-based draws of a candidate's hypothetical outcome.
 *
 * TEST INFRASTRUCTURE ONLY (see fs_oracle.h).
 *
 * Section 4.3 scores a candidate by the expected gap after "revealing its
 * outcome". The paper does not give the posterior inside [lo, hi]; it is
 * read here as a symmetric triangular law (mode at the interval's centre),
 * tabulated at Q equally spaced probabilities and stratified into O equal
 * outcome strata. Both coordinates (capacity, tail) of one scenario fall in
 * the same stratum o and are independent inside it.
 */
#include <math.h>
#include "fs_oracle.h"

/*
 * Philox4x32-10 as defined by Salmon, Moraes, Dror and Shaw, "Parallel
 * Random Numbers: As Easy as 1, 2, 3" (SC'11): ten rounds of a 4x32
 * S-box built from two 32x32->64 multiplications, with a Weyl key
 * schedule. Pinned by the published known-answer vectors
 * (tests/golden/philox4x32_10_kat.txt).
 */
void or_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
    const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
    uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) {
            k0 += W0;
            k1 += W1;
        }
        uint64_t p0 = (uint64_t)M0 * (uint64_t)x0;
        uint64_t p1 = (uint64_t)M1 * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/*
 * Inverse CDF of the symmetric triangular law on [0, 1] at the cell
 * centres u_k = (k + 1/2) / Q. The CDF is 2x^2 below 1/2 and
 * 1 - 2(1-x)^2 above, so x = sqrt(u/2) or 1 - sqrt((1-u)/2). Every step
 * is one correctly rounded float operation (sqrtf is IEEE). Pinned by
 * evaluating the closed-form CDF at each entry in the tests.
 */
void or_triangular_table(int Q, float *qn)
{
    for (int k = 0; k < Q; ++k) {
        float u = ((float)k + 0.5f) / (float)Q;
        float x;
        if (u < 0.5f) {
            x = sqrtf(u * 0.5f);
        } else {
            float v = 1.0f - u;
            x = 1.0f - sqrtf(v * 0.5f);
        }
        qn[k] = x;
    }
}

static int ilog2_exact(int x)
{
    int v = 0;
    while ((1 << v) < x) ++v;
    return ((1 << v) == x) ? v : -1;
}

/*
 * Quantile indices of scenario (cell, o, s). One Philox call serves four
 * consecutive samples: counter (s/4, o, cell, round), key (seed_lo,
 * seed_hi XOR stream_id); sample s takes output word s mod 4. Its upper 16
 * bits give the capacity position and its lower 16 bits the tail position:
 * the top log2(Q/O) bits of each half pick the position inside the outcome
 * stratum [o Q/O, (o+1) Q/O) (Q/O at most 2^16).
 */
int or_draw_index(uint64_t seed, uint32_t stream_id, uint32_t round, int32_t cell,
                  int Q, int O, int o, int s, int32_t *k_cap, int32_t *k_tail)
{
    if (Q < 1 || O < 1 || Q % O != 0) return -1;
    int W = Q / O;
    int w = ilog2_exact(W);
    if (w < 0 || w > 16 || o < 0 || o >= O || s < 0) return -1;
    uint32_t ctr[4] = {(uint32_t)s >> 2, (uint32_t)o, (uint32_t)cell, round};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32) ^ stream_id};
    uint32_t x[4];
    or_philox4x32_10(ctr, key, x);
    uint32_t word = x[s & 3];
    uint32_t hi16 = word >> 16;
    uint32_t lo16 = word & 0xFFFFu;
    *k_cap = o * W + (int32_t)(hi16 >> (16 - w));
    *k_tail = o * W + (int32_t)(lo16 >> (16 - w));
    return 0;
}

/* lo + (hi - lo) q, each step rounded, then clamped to [lo, hi]. */
float or_map(float lo, float hi, float q)
{
    float d = hi - lo;
    float p = d * q;
    float v = lo + p;
    if (v < lo) v = lo;
    if (v > hi) v = hi;
    return v;
}
