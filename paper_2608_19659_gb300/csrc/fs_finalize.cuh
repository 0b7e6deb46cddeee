// Reduction of the fixed-point sums of one problem into E[Gamma_{t+1} | e],
// the score (Section 4.3) and its argmax. Shared by the scorer and the replay.
#pragma once

#include "fs_internal.cuh"

namespace fs {

// Per problem: E[Gamma_{t+1} | e], score, and the argmax (largest score, then
// lower TP = fewer profiling GPU-seconds, then earlier candidate).
struct Best {
  long long sc;
  int j;
  int pos;
};

__device__ __forceinline__ bool better(const Best& a, const Best& b) {
  if (a.pos < 0) return false;
  if (b.pos < 0) return true;
  if (a.sc != b.sc) return a.sc > b.sc;
  if (a.j != b.j) return a.j < b.j;
  return a.pos < b.pos;
}

// (v * 2^-40) / n rounded to the nearest double, for 0 <= v < 2^63 and n >= 1,
// as (double)v * 2^-40 followed by an IEEE division. When n = 2^k the result
// is RN(v) scaled by 2^-(40+k); that double is assembled with integer
// operations (the FP64 unit is narrow on this part): the top 53 significant
// bits of v rounded to nearest, ties to even, and the exponent.
__device__ __forceinline__ double fixed_mean(unsigned long long v, long long n, int log2n) {
  if (log2n < 0) return __ddiv_rn(__dmul_rn(__ll2double_rn((long long)v), 0x1p-40), __ll2double_rn(n));
  if (v == 0ull) return 0.0;
  const int e = 63 - __clzll((long long)v);  // v in [2^e, 2^(e+1))
  unsigned long long m;
  int ex = e;
  if (e <= 52) {
    m = v << (52 - e);
  } else {
    const int sh = e - 52;
    m = v >> sh;
    const unsigned long long rem = v & ((1ull << sh) - 1ull), half = 1ull << (sh - 1);
    if (rem > half || (rem == half && (m & 1ull))) ++m;
    if (m >> 53) {  // rounded up to 2^(e+1)
      m >>= 1;
      ++ex;
    }
  }
  const long long bexp = (long long)ex - 40 - log2n + 1023;  // >= 1023 - 103: a normal double
  return __longlong_as_double((long long)(((unsigned long long)bexp << 52) | (m & ((1ull << 52) - 1ull))));
}

__device__ inline Best finalize_problem(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                                 int p, int beg, int end, double* gap, double* score, float* gt_out) {
  __shared__ Best sb[32];
  const Dims& d = set.d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const float gt = __fsub_rn(set.base[2 * p + 1].t_star, set.base[2 * p].t_star);
  const long long gfix = (long long)fixed40(gt);
  const long long n = (long long)pl.O * pl.S;
  const int log2n = (n & (n - 1)) == 0 ? 63 - __clzll(n) : -1;
  Best b{0, 0, -1};
  for (int q = beg + tid; q < end; q += blockDim.x) {
    long long tot = 0;
#pragma unroll 8
    for (int o = 0; o < pl.O; ++o) tot += (long long)sums[(size_t)q * pl.O + o];
    const long long sc = gfix * n - tot;
    if (gap) gap[q] = fixed_mean((unsigned long long)tot, n, log2n);
    if (score) score[q] = fixed_mean((unsigned long long)sc, n, log2n);
    const Best c{sc, (it.cell[q] / d.B) & 3, q - beg};
    if (better(c, b)) b = c;
  }
  for (int off = 16; off; off >>= 1) {
    Best o;
    o.sc = __shfl_xor_sync(0xffffffffu, b.sc, off);
    o.j = __shfl_xor_sync(0xffffffffu, b.j, off);
    o.pos = __shfl_xor_sync(0xffffffffu, b.pos, off);
    if (better(o, b)) b = o;
  }
  if (lane == 0) sb[warp] = b;
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < nwarp; ++w)
      if (better(sb[w], b)) b = sb[w];
    sb[0] = b;
    if (gt_out) *gt_out = gt;
  }
  __syncthreads();
  return sb[0];
}

}  // namespace fs
