// Allocation solver (Section 3, Eqs. 1-5; tier 2 of the objective) and the
// quantile table, for sm_103a.
//
// One CTA solves one realisation (a capacity and a tail value per cell):
//   1. rows: for every (class i, TP index j) the best SLO-feasible bin
//      (largest capacity, then lowest bin; Eq. 5 gates l <= L_i) -> C_ij.
//      All cells are read once, coalesced; a 32-bit shared-memory atomicMax
//      of the feasible cells' capacity bits per row, then an atomicMin of the
//      bins that hold that capacity (a 64-bit atomicMax of (capacity, -bin)
//      is no native operation: under contention it measured 15x slower);
//   2. thresholds: the positive fulfilments f(n, C_ij), n = 1..floor(G/tau_j)
//      (cut at the first n with f = 1), written to shared memory and
//      bitonic-sorted;
//   3. t*: the largest threshold t whose cheapest per-class covers fit in G.
//      A scoring solve tabulates every row's cover of every threshold (the
//      row table the per-candidate preparation reads) and counts; otherwise a
//      search, each probe one group of lanes (a row per lane, shuffles for the
//      per-class minimum over the four TP lanes and the sum), the groups of the
//      CTA probing evenly spaced points per round;
//   4. choice at t*: per class the cheapest cover, ties to the lower TP.
// For a fixed (TP, n) a larger capacity never lowers f, so the best bin of
// each row is the option the tie rule (larger capacity, then lower bin)
// picks; and t* is the largest threshold t of the rows' values at which the
// total fits, as cost(t) is constant between consecutive thresholds.
// Critical floors (tier 1 of the objective): a row of a critical class i
// starts at its first fulfilment >= delta_i (lower ones are not options), and
// class i covers max(t, delta_i) at threshold t. Step 4 also prices every
// critical class's cheapest cover of its floor: the floors are met when those
// fit in G together; with t* = 0 and the floors met, that cover is the
// class's allocation.
#include <cuda_runtime.h>

#include "fs_internal.cuh"

namespace fs {

__global__ void k_qtable(float* qn, int Q) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= Q) return;
  // Inverse CDF of the symmetric triangular law on [0, 1] at u = (k + 1/2) / Q:
  // 2x^2 = u below 1/2, 1 - 2(1-x)^2 = u above.
  const float u = __fdiv_rn(__fadd_rn(__int2float_rn(k), 0.5f), __int2float_rn(Q));
  float x;
  if (u < 0.5f) {
    x = __fsqrt_rn(__fmul_rn(u, 0.5f));
  } else {
    x = __fsub_rn(1.0f, __fsqrt_rn(__fmul_rn(__fsub_rn(1.0f, u), 0.5f)));
  }
  qn[k] = x;
}

// Total GPUs of the cheapest per-class covers of threshold t (class i covers
// max(t, delta_i)), or kCostInf if some class has no cover, evaluated by an
// aligned group of gsz lanes (a power of two in [4, 32]); lane gl takes rows
// gl, gl + gsz, ... (rho = 4 i + j).
// After the per-class minimum (two xor-shuffles) all four lanes of a class
// hold its cost; xor-sums over the offsets 4 .. gsz/2 then add one lane per
// class, so every lane of the group ends with the total (uncovered classes
// counted above bit 24: a cost is at most G <= 32767, 64 classes < 2^21).
template <bool FL>
__device__ __forceinline__ int group_total_cost(float t, const float* sC, const float* sLam, const float* sRl,
                                                const float* sDl, const Dims& d, int gl, int gsz) {
  int packed = 0;
  for (int base = 0; base < d.K4; base += gsz) {
    const int rho = base + gl;
    int cost = kCostInf;
    if (rho < d.K4) {
      const int j = rho & 3;
      const float tc = FL ? fmaxf(t, sDl[rho >> 2]) : t;
      const int n = min_replicas(tc, sC[rho], sLam[rho >> 2], sRl[rho >> 2], rep_capf(d, j));
      if (n) cost = n << j;
    }
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 1));
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 2));
    int v = rho < d.K4 ? (cost >= kCostInf ? (1 << 24) : cost) : 0;
    for (int off = 4; off < gsz; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    packed += v;
  }
  return (packed >> 24) ? kCostInf : packed;
}

// FL: some class is critical (the model has floors); the instance without floors does
// none of the floor work.
template <bool FL>
__global__ void __launch_bounds__(kSolveThreadsWide) k_solve(Set set, int n_real, const float* cap_x,
                                                         const float* tail_x, fs_allocation* out_x,
                                                         int mode) {
  const bool write_theta = (mode & 1) != 0;
  // the per-class choice at t* (step 4); a scoring call needs only t* and the
  // thresholds, and without floors skips it
  const bool choice = FL || (mode & 2) == 0;
  extern __shared__ __align__(16) unsigned char smraw[];
  const Dims& d = set.d;  // kernel-parameter space: no local copy
  const int r = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_trigger();
  if (r >= n_real) return;

  const float* cap;
  const float* tail;
  int p = 0, sigma = 0;
  fs_allocation* out;
  if (cap_x) {
    cap = cap_x + (size_t)r * d.cells;
    tail = tail_x + (size_t)r * d.cells;
    out = out_x + r;
  } else {
    p = r >> 1;
    sigma = r & 1;
    if (set.skip && set.skip[p] >= 0) return;
    const float* bp = set.bounds + (size_t)p * 4 * d.cells;
    cap = bp + (size_t)(sigma ? CAP_HI : CAP_LO) * d.cells;
    tail = bp + (size_t)(sigma ? TAIL_LO : TAIL_HI) * d.cells;
    out = set.base + r;
  }

  uint32_t* sRowCap = reinterpret_cast<uint32_t*>(smraw);  // [256] best feasible capacity bits per row
  uint32_t* sRowBin = sRowCap + 256;                       // [256] lowest bin holding it (~0u: none)
  float* sC = reinterpret_cast<float*>(sRowBin + 256);    // [256]
  int* sB = reinterpret_cast<int*>(sC + 256);             // [256]
  int* sN0 = sB + 256;                                    // [256]
  int* sOff = sN0 + 256;                                  // [260]
  int* sProbe = sOff + 260;                               // [32]
  int* sMisc = sProbe + 32;                               // [8]
  float* sTheta = reinterpret_cast<float*>(sMisc + 8);    // [pow2 >= theta_cap]

  // 1. rows: the best SLO-feasible bin of each row (largest capacity, then
  // lowest bin). The inputs of the first pass (demands, and each thread's
  // first kPre cells, every cell of a model with at most kPre x 256) are all
  // loaded before anything waits on one of them: one memory round trip. Both
  // passes read those cells from registers; any further cells from memory.
  __shared__ float sLam[FS_MAX_CLASSES], sRl[FS_MAX_CLASSES];  // demand and RN(1/demand)
  __shared__ float sDl[FS_MAX_CLASSES];                          // floor delta_i (0: not critical)
  constexpr int kPre = 4;
  const float lam_v = tid < d.K ? set.lam[tid] : 1.0f;
  const float dl_v = FL && tid < d.K ? set.slo[d.K + tid] : 0.0f;
  float tailp[kPre], capp[kPre], slop[kPre];
#pragma unroll
  for (int k = 0; k < kPre; ++k) {
    const int c = tid + k * (int)blockDim.x;
    const bool in = c < d.cells;
    tailp[k] = in ? tail[c] : 0.0f;
    capp[k] = in ? cap[c] : 0.0f;
    slop[k] = in ? set.slo[(c / d.B) >> 2] : 0.0f;
  }
  for (int rho = tid; rho < d.K4; rho += blockDim.x) {
    sRowCap[rho] = 0u;
    sRowBin[rho] = ~0u;
  }
  if (tid < 8) sMisc[tid] = 0;
  if (tid < d.K) {
    sLam[tid] = lam_v;
    sRl[tid] = __frcp_rn(lam_v);
    if (FL) sDl[tid] = dl_v;
  }
  __syncthreads();
  // feasible cells: their capacity's bits (-0 -> +0: nonnegative floats order
  // like their bit patterns), first the row maximum, then the lowest bin
  // holding it
  bool okp[kPre];
  uint32_t cbp[kPre];
  int rhop[kPre];
#pragma unroll
  for (int k = 0; k < kPre; ++k) {
    const int c = tid + k * (int)blockDim.x;
    rhop[k] = c < d.cells ? c / d.B : 0;
    okp[k] = c < d.cells && tailp[k] <= slop[k];
    cbp[k] = __float_as_uint(__fadd_rn(capp[k], 0.0f));
    if (okp[k]) atomicMax(&sRowCap[rhop[k]], cbp[k]);
  }
  const int c_rest = tid + kPre * (int)blockDim.x;
  for (int c = c_rest; c < d.cells; c += blockDim.x) {
    const int rho = c / d.B;
    if (tail[c] <= set.slo[rho >> 2]) atomicMax(&sRowCap[rho], __float_as_uint(__fadd_rn(cap[c], 0.0f)));
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kPre; ++k) {
    const int c = tid + k * (int)blockDim.x;
    if (okp[k] && cbp[k] == sRowCap[rhop[k]]) atomicMin(&sRowBin[rhop[k]], (uint32_t)(c - rhop[k] * d.B));
  }
  for (int c = c_rest; c < d.cells; c += blockDim.x) {
    const int rho = c / d.B;
    const uint32_t cb = __float_as_uint(__fadd_rn(cap[c], 0.0f));
    if (tail[c] <= set.slo[rho >> 2] && cb == sRowCap[rho]) atomicMin(&sRowBin[rho], (uint32_t)(c - rho * d.B));
  }
  __syncthreads();
  for (int rho = tid; rho < d.K4; rho += blockDim.x) {
    const uint32_t bin = sRowBin[rho];
    const int bb = bin != ~0u ? (int)bin : -1;
    const float best = bb >= 0 ? __uint_as_float(sRowCap[rho]) : 0.0f;
    sC[rho] = best;
    sB[rho] = bb;
    const int i = rho >> 2, j = rho & 3;
    const float lam = sLam[i], rl = sRl[i];
    const int M = rep_cap(d, j);
    const float Mf = rep_capf(d, j);
    int n0 = 0, len = 0;
    if (bb >= 0) {
      atomicOr(reinterpret_cast<unsigned int*>(&sMisc[2 + (i >> 5)]), 1u << (i & 31));
      if (M >= 1) {
        // first fulfilment that is positive and at or above the class's floor
        // (n = 1 unless one replica falls short of it)
        const float lo_f = FL ? fmaxf(sDl[i], __int_as_float(1)) : __int_as_float(1);
        n0 = fulfil_r(1.0f, best, lam, rl) >= lo_f ? 1 : min_replicas(lo_f, best, lam, rl, Mf);
        if (n0) {
          const int ns = min_replicas(1.0f, best, lam, rl, Mf);   // first full fulfilment
          len = ns ? ns : M;
        }
      }
    }
    sN0[rho] = n0;
    sOff[rho] = n0 ? len - n0 + 1 : 0;  // count, scanned below
  }
  __syncthreads();
  if (warp == 0) {  // exclusive scan of the row counts
    int carry = 0;
    for (int base = 0; base < d.K4; base += 32) {
      const int rho = base + lane;
      const int v = rho < d.K4 ? sOff[rho] : 0;
      int incl = v;
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (rho < d.K4) sOff[rho] = carry + incl - v;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) sOff[d.K4] = carry;
  }
  __syncthreads();
  int total = sOff[d.K4];
  if (total > d.theta_cap) {  // cannot happen: a row holds at most floor(G/tau) values
    if (tid == 0) atomicOr(set.status, ST_THETA);
    total = d.theta_cap;
  }
  int P2 = 1;
  while (P2 < total) P2 <<= 1;
  // A scoring solve builds the row table (step 3) when it is small enough; its
  // scratch follows the thresholds: cover costs [K4][total], class minima
  // [K][total], and each row's own fulfilment values in order [total]
  const bool row_table =
      write_theta && !cap_x && set.rtab && d.K4 * total <= kRowTabMax && sOff[d.K4] == total;
  int P2c = 1;
  while (P2c < d.theta_cap) P2c <<= 1;
  int* sCost = reinterpret_cast<int*>(sTheta + P2c);
  int* sCmin = sCost + d.K4 * total;
  float* sOwn = reinterpret_cast<float*>(sCmin + d.K * total);

  // 2. thresholds, then a sort (ascending, +inf padding)
  for (int x = tid; x < P2; x += blockDim.x) {
    float v = __int_as_float(0x7f800000);
    if (x < total) {
      int lo = 0, hi = d.K4 - 1;
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (sOff[mid] <= x) lo = mid; else hi = mid - 1;
      }
      const int n = sN0[lo] + (x - sOff[lo]);
      v = fulfil_r((float)n, sC[lo], sLam[lo >> 2], sRl[lo >> 2]);
      if (row_table) sOwn[x] = v;
    }
    sTheta[x] = v;
  }
  __syncthreads();
  if (P2 <= 64) {
    // small lists: one warp sorts 64 values held two per lane (bitonic network,
    // partners by __shfl_xor_sync), with no block barriers
    if (warp == 0) {
      const float inf = __int_as_float(0x7f800000);
      float r[2] = {lane < P2 ? sTheta[lane] : inf, lane + 32 < P2 ? sTheta[lane + 32] : inf};
      for (int k = 2; k <= 64; k <<= 1) {
        for (int jj = k >> 1; jj > 0; jj >>= 1) {
          if (jj == 32) {  // partners share a lane; k == 64, ascending
            const float lo = fminf(r[0], r[1]), hi = fmaxf(r[0], r[1]);
            r[0] = lo;
            r[1] = hi;
          } else {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int i = lane + 32 * h;
              const float pv = __shfl_xor_sync(0xffffffffu, r[h], jj);
              const bool keep_min = ((i & jj) == 0) == ((i & k) == 0);
              r[h] = keep_min ? fminf(r[h], pv) : fmaxf(r[h], pv);
            }
          }
        }
      }
      if (lane < P2) sTheta[lane] = r[0];
      if (lane + 32 < P2) sTheta[lane + 32] = r[1];
    }
    __syncthreads();
  } else if (row_table && P2 <= 256 && P2 <= (int)blockDim.x) {
    // up to one value a thread, the unsorted values in sOwn: each thread
    // places its value at its rank (values below it, and equal values at
    // lower indices), one pass with no barriers between stages (its cost
    // grows with the count: above 256 values the network below is faster)
    if (tid < total) {
      const float v = sOwn[tid];
      int rank = 0;
#pragma unroll 4
      for (int j = 0; j < total; ++j) {
        const float u = sOwn[j];
        rank += (u < v || (u == v && j < tid)) ? 1 : 0;
      }
      sTheta[rank] = v;
    }
  } else {
    for (int k = 2; k <= P2; k <<= 1) {
      for (int jj = k >> 1; jj > 0; jj >>= 1) {
        for (int x = tid; x < P2; x += blockDim.x) {
          const int y = x ^ jj;
          if (y > x) {
            const float a = sTheta[x], b = sTheta[y];
            const bool up = (x & k) == 0;
            if ((a > b) == up && a != b) {
              sTheta[x] = b;
              sTheta[y] = a;
            }
          }
        }
        __syncthreads();
      }
    }
  }

  // 3. t*: the largest index whose threshold fits in G (the cheapest-cover
  // total is nondecreasing along the sorted thresholds).
  __shared__ int s_res[2][kSolveThreadsWide / 4];
  if (tid == 0) sMisc[4] = 0;
  __syncthreads();
  int kstar;
  if (row_table) {
    // Row table of a scoring solve: every row's cover cost at every threshold,
    // then per (row rho, threshold k) the word the per-candidate preparation
    // reads for a candidate in row rho, stored threshold-major at k K4 + rho (its
    // address does not depend on the number of thresholds): bits 0-15 the
    // replicas rho may use once the other classes are covered (0 if one cannot
    // be), bit 16 set if another row of rho's class covers theta_k within that
    // budget.
    //
    // A row's cheapest cover of t (class i covers max(t, delta_i)) is n0 plus
    // the number of its own values f(n0) <= ... <= f(len) below t: every n
    // below n0 falls short of it, and past len either f(ns) >= 1 >= t or the
    // row holds M replicas and none covers t. The values are the fulfilments
    // the thresholds were made of, so the count is the cover min_replicas
    // finds, without evaluating f. One thread per (class, threshold) runs the
    // four TP rows' branch-free lower bounds side by side.
    const int nx = d.K * total;
    for (int x = tid; x < nx; x += blockDim.x) {
      const int i = x / total, k = x - i * total;
      const float tc = FL ? fmaxf(sTheta[k], sDl[i]) : sTheta[k];
      int q[4], nv[4], beg[4];  // values below tc so far, values held, first value
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        beg[j] = sOff[4 * i + j];
        nv[j] = sOff[4 * i + j + 1] - beg[j];
        q[j] = 0;
      }
      const int most = max(max(nv[0], nv[1]), max(nv[2], nv[3]));
      for (int step = most ? 1 << (31 - __clz(most)) : 0; step > 0; step >>= 1) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          // the four loads are issued unconditionally: the index is clamped to
          // the row's last value, at most total - 1 (an empty row reads the word
          // before its start, at worst the last class minimum: scratch either way)
          const float v = sOwn[beg[j] + min(q[j] + step, nv[j]) - 1];
          q[j] += (q[j] + step <= nv[j]) & (v < tc) ? step : 0;
        }
      }
      int cm = kCostInf;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = q[j] < nv[j] ? (sN0[4 * i + j] + q[j]) << j : kCostInf;
        sCost[(4 * i + j) * total + k] = c;
        cm = min(cm, c);
      }
      sCmin[x] = cm;
    }
    __syncthreads();
    // per pair: the other classes' covers summed (an uncovered class counted as
    // 2^24: a cost is at most G <= 32767, 64 of them stay below 2^21), then one
    // word per TP row; t* = the count of thresholds whose total fits, less one
    int* rt = set.rtab + ((size_t)p * 2 + sigma) * kRowTabMax;
    int cnt = 0;
    for (int x0 = 0; x0 < nx; x0 += blockDim.x) {
      const int x = x0 + tid;
      bool fits = false;
      if (x < nx) {
        const int i = x / total, k = x - i * total;
        int sum = 0;
        for (int q = 0; q < d.K; ++q) {
          const int cq = sCmin[q * total + k];
          sum += cq >= kCostInf ? (1 << 24) : cq;
        }
        fits = i == 0 && sum <= d.G;
        const int own = sCmin[x];
        const int rest = sum - (own >= kCostInf ? (1 << 24) : own);
        const int A = (rest >> 24) ? -1 : d.G - rest;
        int c[4], wd[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) c[j] = sCost[(4 * i + j) * total + k];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          int other = kCostInf;  // cheapest cover by another row of the class
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (q != j) other = min(other, c[q]);
          const int m = A >= (1 << j) ? min(A >> j, rep_cap(d, j)) : 0;
          wd[j] = m | ((other < kCostInf && other <= A) ? 1 << 16 : 0);
        }
        // threshold-major: word (rho, k) at k K4 + rho, the class's four in one 16-byte store
        *reinterpret_cast<int4*>(rt + (size_t)k * d.K4 + 4 * i) = make_int4(wd[0], wd[1], wd[2], wd[3]);
      }
      cnt += __syncthreads_count(fits);
    }
    kstar = cnt - 1;
  } else {
    // Search: each round every group of gsz lanes probes one index (an
    // (ng+1)-ary split); each warp merges the answers with integer max / min
    // reductions, so a round costs one barrier (lo feasible, hi not).
    int gsz = 4;
    while (gsz < d.K4 && gsz < 32) gsz <<= 1;
    const int ng = blockDim.x / gsz, g = tid / gsz, gl = tid & (gsz - 1);
    int lo = -1, hi = total;
    for (int par = 0; hi - lo > 1; par ^= 1) {
      int kp = lo + ((g + 1) * (hi - lo)) / (ng + 1);
      kp = max(lo + 1, min(hi - 1, kp));
      const int cost = group_total_cost<FL>(sTheta[kp], sC, sLam, sRl, sDl, d, gl, gsz);
      if (gl == 0) s_res[par][g] = (cost <= d.G) ? kp : -(kp + 1);
      __syncthreads();
      int nlo = lo, nhi = hi;
      for (int q = lane; q < ng; q += 32) {
        const int v = s_res[par][q];
        if (v >= 0) nlo = max(nlo, v); else nhi = min(nhi, -v - 1);
      }
      lo = __reduce_max_sync(0xffffffffu, nlo);
      hi = __reduce_min_sync(0xffffffffu, nhi);
    }
    kstar = lo;
  }
  const float tstar = kstar >= 0 ? sTheta[kstar] : 0.0f;

  if (choice) {
    // 4. choice at t*: every row's cheapest cover in parallel (thread = row), then
    // per class the cheapest row over its four TP lanes, lower TP on ties; the
    // same for the floor of a critical class, summed into sMisc[5] (sMisc[6]:
    // some critical class cannot reach its floor)
    {
      const int rho = tid;  // K4 <= 256 <= blockDim
      int key = 0x7fffffff, keyf = 0x7fffffff;
      if (rho < d.K4) {
        const float dl = FL ? sDl[rho >> 2] : 0.0f;
        if (tstar > 0.0f) {
          const int n = min_replicas(FL ? fmaxf(tstar, dl) : tstar, sC[rho], sLam[rho >> 2], sRl[rho >> 2],
                                     rep_capf(d, rho & 3));
          if (n) key = ((n << (rho & 3)) << 2) | (rho & 3);
        }
        if (FL && dl > 0.0f) {
          const int n = min_replicas(dl, sC[rho], sLam[rho >> 2], sRl[rho >> 2], rep_capf(d, rho & 3));
          if (n) keyf = ((n << (rho & 3)) << 2) | (rho & 3);
        }
      }
      key = min(key, __shfl_xor_sync(0xffffffffu, key, 1));
      key = min(key, __shfl_xor_sync(0xffffffffu, key, 2));
      const int i = tid >> 2;
      if constexpr (FL) {
        keyf = min(keyf, __shfl_xor_sync(0xffffffffu, keyf, 1));
        keyf = min(keyf, __shfl_xor_sync(0xffffffffu, keyf, 2));
        const bool critical = (tid & 3) == 0 && i < d.K && sDl[i] > 0.0f;
        if (critical) {
          if (keyf == 0x7fffffff) atomicOr(&sMisc[6], 1);
          else atomicAdd(&sMisc[5], keyf >> 2);
        }
        __syncthreads();
        const bool met = sMisc[6] == 0 && sMisc[5] <= d.G;
        if (tstar <= 0.0f) key = (critical && met) ? keyf : 0x7fffffff;  // tier 1 alone
      }
      if ((tid & 3) == 0 && i < FS_MAX_CLASSES) {  // (a 512-thread block has 128 groups of four)
        int8_t tp = 0;
        int16_t bin = -1, reps = 0;
        float f = 0.0f;
        if (i < d.K && key != 0x7fffffff) {
          const int bj = key & 3, cost_i = key >> 2, bn = cost_i >> bj;
          tp = (int8_t)(1 << bj);
          bin = (int16_t)sB[4 * i + bj];
          reps = (int16_t)bn;
          f = fulfil_r((float)bn, sC[4 * i + bj], sLam[i], sRl[i]);
          atomicAdd(&sMisc[4], cost_i);
        }
        out->tp[i] = tp;
        out->bin[i] = bin;
        out->replicas[i] = reps;
        out->fulfil[i] = f;
      }
    }
    __syncthreads();
  }
  if (tid == 0) {
    out->t_star = tstar;
    // (with t* = 0 and no floors the sum is 0 anyway; the unconditional read
    // measured 1.5 us slower on a 28 us scoring call whose next kernel overlaps this one)
    out->total_gpus = !choice ? -1 : (FL || tstar > 0.0f) ? sMisc[4] : 0;  // -1: not computed
    out->has_option_mask = (uint64_t)(uint32_t)sMisc[2] | ((uint64_t)(uint32_t)sMisc[3] << 32);
    out->ok = tstar > 0.0f ? 1 : 0;
    out->floors_met = (!FL || (sMisc[6] == 0 && sMisc[5] <= d.G)) ? 1 : 0;
    out->goodput = 0.0;  // tier 3 is filled by the lexicographic solve
  }
  if (write_theta && !cap_x) {
    float* th = set.theta + ((size_t)p * 2 + sigma) * d.theta_cap;
    for (int x = tid; x < total; x += blockDim.x) th[x] = sTheta[x];
    float* rc = set.rowC + ((size_t)p * 2 + sigma) * d.K4;
    int* rb = set.rowB + ((size_t)p * 2 + sigma) * d.K4;
    for (int rho = tid; rho < d.K4; rho += blockDim.x) {
      rc[rho] = sC[rho];
      rb[rho] = sB[rho];
    }
    if (tid == 0) set.ntheta[p * 2 + sigma] = total;
  }
}

// Watchdog self-test: wait on a barrier phase that nothing completes; the
// bounded wait gives up, records the timeout and the kernel returns.
__global__ void k_watchdog(uint32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) mbar_init(&bar, 1);
  __syncthreads();
  const bool ok = mbar_wait(&bar, 0u, limit_ns);
  if (!ok && threadIdx.x == 0) atomicOr(status, ST_TIMEOUT);
}

cudaError_t launch_watchdog(uint32_t* status, uint64_t limit_ns, cudaStream_t s) {
  note_launch();
  k_watchdog<<<1, 32, 0, s>>>(status, limit_ns);
  return cudaGetLastError();
}

static size_t solve_smem_bytes(const Dims& d) {
  int P2 = 1;
  while (P2 < d.theta_cap) P2 <<= 1;
  return 256 * 8 + (size_t)(256 * 3 + 260 + 32 + 8) * 4 + (size_t)P2 * 4;
}

cudaError_t launch_qtable(float* qn, int Q, cudaStream_t s) {
  note_launch();
  k_qtable<<<(Q + 255) / 256, 256, 0, s>>>(qn, Q);
  return cudaGetLastError();
}

cudaError_t launch_solve(const Set& set, int n, const float* cap_x, const float* tail_x,
                         fs_allocation* out, bool write_theta, LaunchCache& lc, cudaStream_t s, bool tstar_only) {
  if (n <= 0) return cudaSuccess;
  // a scoring solve may build the row table: K4 x |Theta| cover costs, K x |Theta| class minima
  // and |Theta| own values, with K4 x |Theta| <= kRowTabMax
  const size_t smem =
      solve_smem_bytes(set.d) + (write_theta && set.rtab ? (size_t)(kRowTabMax + kRowTabMax / 2) * 4 : 0);
  const int fl = lc.floors ? 1 : 0;
  auto kern = fl ? k_solve<true> : k_solve<false>;
  if (smem > lc.solve_smem[fl]) {
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), smem);
    if (e != cudaSuccess) return e;
    lc.solve_smem[fl] = smem;
  }
  // a scoring solve of a model with more than 256 cells takes 512 threads: its
  // per-cell passes and row-table phases then run half the iterations each
  const int bt = write_theta && !cap_x && set.d.cells > kSolveThreads ? kSolveThreadsWide : kSolveThreads;
  note_launch();
  kern<<<n, bt, smem, s>>>(set, n, cap_x, tail_x, out, (write_theta ? 1 : 0) | (tstar_only ? 2 : 0));
  return cudaGetLastError();
}

}  // namespace fs
