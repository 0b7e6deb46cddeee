// Reduction of the fixed-point sums of one problem into E[Gamma_{t+1} | e],
// the score (Section 4.3) and its argmax. Shared by the scorer and the replay.
#pragma once

#include "fs_internal.cuh"

namespace fs {

// Per problem: E[Gamma_{t+1} | e], score, and the argmax (largest score, then
// lower TP = fewer profiling GPU-seconds, then earlier candidate). The order
// is carried as a key compared without branches: hi = the score's fixed-point
// value (the smallest int64 for "no candidate"), lo = (3 - j) 2^30 +
// (2^30 - 1 - pos), larger is better in both (pos < 2^30: n_cand O <= 2^30).
constexpr long long kNoScore = (-0x7FFFFFFFFFFFFFFFLL - 1);

struct Best {
  long long hi;
  uint32_t lo;
  int cell;  // the candidate's cell, carried so that no load follows the reduction
  __device__ __forceinline__ bool valid() const { return hi != kNoScore; }
  __device__ __forceinline__ int pos() const { return (int)(0x3FFFFFFFu - (lo & 0x3FFFFFFFu)); }
};

__device__ __forceinline__ Best make_best(long long sc, int j, int pos, int cell) {
  return Best{sc, ((uint32_t)(3 - j) << 30) | (0x3FFFFFFFu - (uint32_t)pos), cell};
}

__device__ __forceinline__ Best no_best() { return Best{kNoScore, 0u, -1}; }

__device__ __forceinline__ bool better(const Best& a, const Best& b) {
  return a.hi > b.hi || (a.hi == b.hi && a.lo > b.lo);
}

// The best of the 32 lanes' values (butterfly over xor-shuffles: every lane
// ends with it).
__device__ __forceinline__ Best warp_best(Best b) {
  for (int off = 16; off; off >>= 1) {
    Best o;
    o.hi = __shfl_xor_sync(0xffffffffu, b.hi, off);
    o.lo = __shfl_xor_sync(0xffffffffu, b.lo, off);
    o.cell = __shfl_xor_sync(0xffffffffu, b.cell, off);
    const bool t = better(o, b);
    b.hi = t ? o.hi : b.hi;
    b.lo = t ? o.lo : b.lo;
    b.cell = t ? o.cell : b.cell;
  }
  return b;
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

// Items [beg, end) of problem p, whose first item is pos0 (candidate positions,
// for the order of equal scores, count from there).
__device__ inline Best finalize_problem(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                                 int p, int beg, int end, double* gap, double* score, float* gt_out,
                                 int pos0) {
  __shared__ Best sb[32];
  const Dims& d = set.d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  // inputs are read-only here (written by earlier kernels): every load goes
  // through the read-only path and is issued before any store
  const float gt = __fsub_rn(__ldg(&set.base[2 * p + 1].t_star), __ldg(&set.base[2 * p].t_star));
  const long long gfix = (long long)fixed40(gt);
  const long long n = (long long)pl.O * pl.S;
  const int log2n = (n & (n - 1)) == 0 ? 63 - __clzll(n) : -1;
  Best b = no_best();
  for (int q = beg + tid; q < end; q += blockDim.x) {
    const int cell = __ldg(it.cell + q);
    long long tot = 0;
#pragma unroll 8
    for (int o = 0; o < pl.O; ++o) tot += (long long)__ldg(sums + (size_t)q * pl.O + o);
    const long long sc = gfix * n - tot;
    if (gap) gap[q] = fixed_mean((unsigned long long)tot, n, log2n);
    if (score) score[q] = fixed_mean((unsigned long long)sc, n, log2n);
    const Best c = make_best(sc, (cell / d.B) & 3, q - pos0, cell);
    if (better(c, b)) b = c;
  }
  b = warp_best(b);
  if (lane == 0) sb[warp] = b;
  __syncthreads();
  if (warp == 0) {  // the warps' results, reduced by warp 0 in parallel
    b = warp_best(lane < nwarp ? sb[lane] : no_best());
    if (lane == 0) {
      sb[0] = b;
      if (gt_out) *gt_out = gt;
    }
  }
  __syncthreads();
  return sb[0];
}

}  // namespace fs
