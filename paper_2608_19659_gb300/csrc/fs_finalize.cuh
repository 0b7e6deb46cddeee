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

__device__ inline Best finalize_problem(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                                 int p, int beg, int end, double* gap, double* score, float* gt_out) {
  __shared__ Best sb[32];
  const Dims& d = set.d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const float gt = __fsub_rn(set.base[2 * p + 1].t_star, set.base[2 * p].t_star);
  const long long gfix = __float2ll_rn(__fmul_rn(gt, 0x1p40f));
  const long long n = (long long)pl.O * pl.S;
  Best b{0, 0, -1};
  for (int q = beg + tid; q < end; q += blockDim.x) {
    long long tot = 0;
    for (int o = 0; o < pl.O; ++o) tot += (long long)sums[(size_t)q * pl.O + o];
    const long long sc = gfix * n - tot;
    if (gap) gap[q] = __ddiv_rn(__dmul_rn(__ll2double_rn(tot), 0x1p-40), __ll2double_rn(n));
    if (score) score[q] = __ddiv_rn(__dmul_rn(__ll2double_rn(sc), 0x1p-40), __ll2double_rn(n));
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
