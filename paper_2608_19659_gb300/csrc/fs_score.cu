// Monte-Carlo decision-gap scorer (Section 4.3) for sm_103a.
//
// score_t(e) = E[Gamma_t - Gamma_{t+1} | e] with Gamma = t*(A+) - t*(A-)
// (Sections 4.1-4.2). A scenario (e, o, s) draws (c_y, l_y) for cell e and
// re-solves both realisations with cell e replaced. Only row r = (i_e, j_e)
// changes, and only through its best capacity
//     C' = (l_y <= L_i) ? max(Cexcl, c_y) : Cexcl,
// where Cexcl is the best SLO-feasible capacity of the row's other bins
// under the same realisation. The scenario solve is therefore parametric in
// the scalar C':
//
//   For a threshold t of the realisation's sorted threshold set Theta, let
//   A(t) = G - sum_{i != i_e} cost_i(t) be the budget left for class i_e and
//   P(t) its cheapest cover without row r. t is feasible with row capacity C'
//   iff P(t) <= A(t) or f(m(t), C') >= t, where m(t) = min(floor(A/tau_r),
//   floor(G/tau_r)); feasibility is monotone in t, so
//   kappa(t) = min{C' : t feasible} is nondecreasing along Theta.
//   With b = the last index with kappa <= C' (theta_b = 0 if none),
//   t* = max(theta_b, f(m(theta_{b+1}), C'))   (the second term only if > theta_b):
//   between theta_b and theta_{b+1} the other classes' costs are constant, so
//   the best cover by row r alone is its largest fulfilment within budget.
//   Theta may contain values of row r itself (a superset is harmless).
//   Critical floors (tier 1): class i covers max(t, delta_i) at threshold t,
//   the base thresholds already leave out values below a floor, and row r's
//   own term counts only at or above delta_{i_e}.
//
// k_prep builds, per (candidate, realisation), the part of that table a
// scenario can reach: Theta entries with kappa in (Cexcl, max(Cexcl, cap_hi_e)].
// m(t) and "P(t) <= A(t)" depend only on (r, t): a scoring solve tabulates
// them per realisation (the row table, k_solve), and k_prep then finds the
// range's ends as counts of feasible thresholds and each kappa by one thread;
// without a table it searches, evaluating the rows per probe.
// It also maps each outcome's quantile stratum into the candidate's capacity
// interval and records where the stratum's tail values stop passing the SLO
// (the map is monotone, so the gate of Eq. 5 is a position test).
// k_score draws each scenario (Philox4x32-10 + quantile lookup), evaluates
// both t* by a binary search of the staged table plus one fulfilment, and
// sums g = rint(Gamma' 2^40) in int64. k_finalize turns the sums into
// E[Gamma_{t+1} | e], the score and the argmax.
#include <cuda_runtime.h>

#include <algorithm>
#include <vector>

#include "fs_finalize.cuh"
#include "fs_internal.cuh"
#include "fs_sample.cuh"

namespace fs {

// Budget left for class ie and its cheapest cover without row rr, at threshold t.
struct Eval {
  int A;   // -1 if another class has no cover
  int P;   // kCostInf if no other row of class ie covers t
};

// Evaluation of threshold t by an aligned group of gsz lanes (gsz a power of
// two in [4, 32]); lane gl of the group takes rows gl, gl + gsz, ... The
// per-class minimum over the four TP rows is two xor-shuffles, after which all
// four lanes of a class hold its cost; xor-sums over the offsets 4 .. gsz/2
// then add one lane of every class, so every lane of the group ends with the
// other classes' total (uncovered classes counted above bit 24: a cost is at
// most G <= 32767, so 64 of them stay below 2^21), and every lane's result is valid.
template <bool FL>
__device__ __forceinline__ Eval group_eval_excl(float t, const float* sC, const float* sLam, const float* sRl,
                                                const float* sDl, const Dims& d, int rr, int ie, int gl, int gsz) {
  int packed = 0;
  int P = kCostInf;
  for (int base = 0; base < d.K4; base += gsz) {
    const int rho = base + gl;
    int cost = kCostInf;
    if (rho < d.K4 && rho != rr) {
      const float tc = FL ? fmaxf(t, sDl[rho >> 2]) : t;
      const int n = min_replicas(tc, sC[rho], sLam[rho >> 2], sRl[rho >> 2], rep_capf(d, rho & 3));
      if (n) cost = n << (rho & 3);
    }
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 1));
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 2));
    const bool other = rho < d.K4 && (rho >> 2) != ie;
    int v = other ? (cost >= kCostInf ? (1 << 24) : cost) : 0;
    for (int off = 4; off < gsz; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    packed += v;
    const int ib = ie * 4;
    const int pc = __shfl_sync(0xffffffffu, cost, (ib - base) & (gsz - 1), gsz);
    if (ib >= base && ib < base + gsz) P = pc;
  }
  Eval e;
  e.A = (packed >> 24) ? -1 : d.G - packed;
  e.P = P;
  return e;
}

__device__ __forceinline__ int replicas_left(const Eval& e, int jr, const Dims& d) {
  return (e.A >= (1 << jr)) ? min(e.A >> jr, rep_cap(d, jr)) : 0;
}

// te = max(t, delta_{i_e}): the fulfilment row r must reach
__device__ __forceinline__ bool feasible_at(const Eval& e, int m, float C, float te, float lam, float rl) {
  return (e.P < kCostInf && e.P <= e.A) || (m >= 1 && fulfil_r((float)m, C, lam, rl) >= te);
}

// Index probed by group g of ng in one round of the joint search for the
// last feasible index at Cexcl (interval (lo0, hi0)) and at max(Cexcl,
// cap_hi) (interval (lo1, hi1)); open intervals are split evenly.
__device__ __forceinline__ int probe_index(int g, int ng, int lo0, int hi0, int lo1, int hi1) {
  const bool open0 = hi0 - lo0 > 1, open1 = hi1 - lo1 > 1;
  int lo, hi, part, parts;
  if (open0 && open1) {
    const int half = ng >> 1;
    const bool first = g < half;
    lo = first ? lo0 : lo1;
    hi = first ? hi0 : hi1;
    parts = half + 1;
    part = (first ? g : g - half) + 1;
  } else {
    lo = open0 ? lo0 : lo1;
    hi = open0 ? hi0 : hi1;
    parts = ng + 1;
    part = g + 1;
  }
  const int k = lo + (part * (hi - lo)) / parts;
  return max(lo + 1, min(hi - 1, k));
}

// Smallest bit pattern C in (bx, bmax] with fulfil(m, C) >= t, given that bmax
// qualifies (fulfil is nondecreasing in C, and nonnegative floats order like
// their bit patterns). From the estimate `guess` it gallops (steps 1, 2, 4,
// ...) until the answer is bracketed, then bisects: a few evaluations when the
// estimate is within a few units in the last place, at most about 64 for any.
__device__ __forceinline__ uint32_t kappa_walk(float mf, float t, float lam, float rl, uint32_t bx,
                                               uint32_t bmax, uint32_t guess) {
  uint32_t lo = bx, hi = bmax;  // lo fails (or is Cexcl itself), hi passes
  const uint32_t g = min(max(guess, bx + 1u), bmax);
  const bool up = g < bmax && fulfil_r(mf, __uint_as_float(g), lam, rl) < t;
  if (up) lo = g; else hi = g;
  for (uint32_t step = 1; hi - lo > 1; step <<= 1) {
    const uint32_t w = min(step, hi - lo - 1);
    const uint32_t q = up ? lo + w : hi - w;
    const bool ok = fulfil_r(mf, __uint_as_float(q), lam, rl) >= t;
    if (ok) hi = q; else lo = q;
    if (ok == up) break;  // bracketed
  }
  while (hi - lo > 1) {
    const uint32_t mid = lo + ((hi - lo) >> 1);
    if (fulfil_r(mf, __uint_as_float(mid), lam, rl) >= t) hi = mid; else lo = mid;
  }
  return hi;
}

// t* of one realisation with row capacity C (defined below, with the scorer).
template <int ROW, bool FL>
__device__ __forceinline__ float tstar_of(float C, const float* kap, const float* thx, const float* mnx,
                                          int step0, float lam, float rlam, float dl);

// One CTA per (candidate, realisation sigma). Before the threshold search it
// maps the quantile strata of the outcomes o = sigma, sigma + 2, ... into the
// candidate's record: this and Cexcl read only the bounds, so with `early`
// they overlap the base solve that precedes this kernel. FL: some class is
// critical (the model has floors).
template <bool FL, bool RF>
__global__ void __launch_bounds__(kPrepThreads) k_prep(Set set, Items it, Plan pl, float* rec,
                                                       uint64_t* sums, int early, int th_cap) {
  extern __shared__ __align__(16) unsigned char smraw[];
  float* sC = reinterpret_cast<float*>(smraw);  // [256]
  float* sTh = sC + 256;                          // [th_cap]
  __shared__ float s_cx, s_cmax, s_pc, s_po, s_lf, s_hf;
  __shared__ int s_bx, s_row;
  __shared__ float sLam[FS_MAX_CLASSES], sRl[FS_MAX_CLASSES];  // demand and RN(1/demand)
  __shared__ float sDl[FS_MAX_CLASSES];                          // floor delta_i (0: not critical)
  __shared__ int s_res[2][kPrepThreads / 4];
  const Dims& d = set.d;  // kernel-parameter space: no local copy
  const int item = blockIdx.x >> 1, sigma = blockIdx.x & 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  if (!early) pdl_wait();
  const int p = it.p ? it.p[item] : 0;
  const int cell = it.cell[item];
  float* base_rec = rec + (size_t)item * pl.item_floats;
  float* tab = base_rec + (size_t)sigma * d.slot_floats;
  if (blockIdx.x == 0 && tid == 0) {
    set.work[0] = 0ull;  // the Monte-Carlo kernel's chunk counter
    set.work[1] = 0ull;  // the reduction's ticket
  }
  if (sigma == 0)
    for (int o = tid; o < pl.O; o += blockDim.x) sums[(size_t)item * pl.O + o] = 0ull;
  if (cell < 0 || cell >= d.cells) {  // device-side candidate ids are checked here
    if (tid == 0) {
      atomicOr(set.status, ST_CELL);
      for (int k = 0; k < kTableHeader; ++k) tab[k] = 0.0f;
      tab[H_BX] = __int_as_float(-1);
      tab[H_CELL] = __int_as_float(-1);
    }
    return;
  }
  const int rr = cell / d.B, be = cell - rr * d.B, ie = rr >> 2, jr = rr & 3;
  const float lam = set.lam[ie], L = set.slo[ie], rl = __frcp_rn(lam);
  const float dle = FL ? set.slo[d.K + ie] : 0.0f;
  if (tid < d.K) {
    sLam[tid] = set.lam[tid];
    sRl[tid] = __frcp_rn(set.lam[tid]);
    if (FL) sDl[tid] = set.slo[d.K + tid];
  }
  const float* bp = set.bounds + (size_t)p * 4 * d.cells;
  const float* capS = bp + (size_t)(sigma ? CAP_HI : CAP_LO) * d.cells;
  const float* tailS = bp + (size_t)(sigma ? TAIL_LO : TAIL_HI) * d.cells;
  const float lo_c = bp[(size_t)CAP_LO * d.cells + cell], hi_c = bp[(size_t)CAP_HI * d.cells + cell];
  const float lo_l = bp[(size_t)TAIL_LO * d.cells + cell], hi_l = bp[(size_t)TAIL_HI * d.cells + cell];

  // best SLO-feasible capacity of row r without bin b_e (ties: lower bin)
  if (RF) {
    // Under the monotone prior a scenario's draw (c_y, l_y) also refits row
    // r's other bins (capacity and tail nondecreasing in the load bin). For
    // realisation sigma the row's capacity is then
    //   C' = max(g ? max(P_open, c_y) : P_closed, min(max(c_y, F_lo), F_hi)):
    // A- (sigma 0): a bin below b_e keeps cap_lo and its upper tail falls to
    //   max(min(tail_hi, l_y), tail_lo), which passes the SLO iff tail_hi <= L,
    //   or g and tail_lo <= L (P); a bin above b_e passes iff tail_hi <= L and
    //   its lower capacity rises to min(max(cap_lo, c_y), cap_hi), whose
    //   maximum over such bins is min(max(c_y, max cap_lo), max cap_hi) (F).
    // A+ (sigma 1): a bin above b_e keeps cap_hi and its lower tail rises to
    //   min(max(tail_lo, l_y), tail_hi), which passes iff tail_hi <= L, or g
    //   and tail_lo <= L (P); a bin below b_e passes iff tail_lo <= L and its
    //   upper capacity falls to max(min(cap_hi, c_y), cap_lo) (F).
    // So C' depends on the draw only through (c_y, g), as without the prior.
    if (warp == 0) {
      float pc = 0.0f, po = 0.0f, lf = 0.0f, hf = 0.0f;
      const float* cl = bp + (size_t)CAP_LO * d.cells + (size_t)rr * d.B;
      const float* ch = bp + (size_t)CAP_HI * d.cells + (size_t)rr * d.B;
      const float* tl = bp + (size_t)TAIL_LO * d.cells + (size_t)rr * d.B;
      const float* th = bp + (size_t)TAIL_HI * d.cells + (size_t)rr * d.B;
      for (int b = lane; b < d.B; b += 32) {
        if (b == be) continue;
        const bool p_side = sigma ? b > be : b < be;  // bins refit only in their tail
        const float cap = sigma ? ch[b] : cl[b];
        if (p_side) {
          if (th[b] <= L) pc = fmaxf(pc, cap);
          if (tl[b] <= L) po = fmaxf(po, cap);
        } else if ((sigma ? tl[b] : th[b]) <= L) {  // bins refit only in their capacity
          lf = fmaxf(lf, cl[b]);
          hf = fmaxf(hf, ch[b]);
        }
      }
      for (int off = 16; off; off >>= 1) {
        pc = fmaxf(pc, __shfl_xor_sync(0xffffffffu, pc, off));
        po = fmaxf(po, __shfl_xor_sync(0xffffffffu, po, off));
        lf = fmaxf(lf, __shfl_xor_sync(0xffffffffu, lf, off));
        hf = fmaxf(hf, __shfl_xor_sync(0xffffffffu, hf, off));
      }
      if (lane == 0) {
        po = fmaxf(po, pc);
        // the table covers C' from its least (c_y = cap_lo, gate closed) to
        // its largest value (c_y = cap_hi, gate open)
        s_cx = fmaxf(pc, fminf(fmaxf(lo_c, lf), hf));
        s_cmax = fmaxf(fmaxf(po, hi_c), fminf(fmaxf(hi_c, lf), hf));
        s_pc = pc;
        s_po = po;
        s_lf = lf;
        s_hf = hf;
        s_bx = -1;
        s_row = 0;
      }
    }
  } else if (warp == 0) {
    float best = 0.0f;
    int bb = -1;
    for (int b = lane; b < d.B; b += 32) {
      if (b == be) continue;
      const size_t c = (size_t)rr * d.B + b;
      if (tailS[c] <= L) {
        const float v = capS[c];
        if (bb < 0 || v > best) {
          best = v;
          bb = b;
        }
      }
    }
    for (int off = 16; off; off >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, off);
      const int obb = __shfl_xor_sync(0xffffffffu, bb, off);
      if (obb >= 0 && (bb < 0 || ob > best || (ob == best && obb < bb))) {
        best = ob;
        bb = obb;
      }
    }
    if (lane == 0) {
      s_cx = bb >= 0 ? best : 0.0f;
      s_bx = bb;
      s_cmax = fmaxf(s_cx, hi_c);
      s_pc = s_po = s_cx;
      s_lf = s_hf = 0.0f;
      s_row = 0;
    }
  }

  // Mapped strata. Window of outcome o: word 0 = the number of leading
  // positions whose tail value passes the SLO (the mapped tails are
  // nondecreasing in the position, so exactly one position ends the run of
  // passes), words 4.. = the W capacities.
  {
    const int W = pl.W;
    const float d_c = __fsub_rn(hi_c, lo_c), d_l = __fsub_rn(hi_l, lo_l);
    const long long n_idx = (long long)((pl.O - sigma + 1) >> 1) * W;
    float* wins = base_rec + 2 * (size_t)d.slot_floats;
    if (W >= 4 && (reinterpret_cast<uintptr_t>(set.qn) & 15u) == 0) {
      // four consecutive positions per thread: one 16-byte load and store
      // (windows start on 16-byte boundaries), plus the next position's value
      const long long n4 = n_idx >> 2;
#pragma unroll 2
      for (long long g4 = tid; g4 < n4; g4 += blockDim.x) {
        const long long idx = g4 << 2;
        const int k = (int)(idx & (W - 1));
        const int o = sigma + 2 * (int)(idx >> pl.w);
        const float* q = set.qn + (size_t)o * W;
        float* win = wins + (size_t)o * pl.Wp;
        const float4 v = __ldg(reinterpret_cast<const float4*>(q + k));
        const float vn = k + 4 < W ? __ldg(q + k + 4) : 0.0f;
        float4 cm;
        cm.x = map_into(lo_c, d_c, hi_c, v.x);
        cm.y = map_into(lo_c, d_c, hi_c, v.y);
        cm.z = map_into(lo_c, d_c, hi_c, v.z);
        cm.w = map_into(lo_c, d_c, hi_c, v.w);
        *reinterpret_cast<float4*>(win + 4 + k) = cm;
        const bool p0 = map_into(lo_l, d_l, hi_l, v.x) <= L, p1 = map_into(lo_l, d_l, hi_l, v.y) <= L;
        const bool p2 = map_into(lo_l, d_l, hi_l, v.z) <= L, p3 = map_into(lo_l, d_l, hi_l, v.w) <= L;
        const bool p4 = k + 4 < W && map_into(lo_l, d_l, hi_l, vn) <= L;
        if (k == 0 && !p0) win[0] = __int_as_float(0);
        if (p0 && !p1) win[0] = __int_as_float(k + 1);
        if (p1 && !p2) win[0] = __int_as_float(k + 2);
        if (p2 && !p3) win[0] = __int_as_float(k + 3);
        if (p3 && !p4) win[0] = __int_as_float(k + 4);
      }
    } else {
      // read-only loads, so that the unrolled iterations' loads are issued
      // together rather than each behind the previous iteration's stores
#pragma unroll 4
      for (long long idx = tid; idx < n_idx; idx += blockDim.x) {
        const int k = (int)(idx & (W - 1));
        const int o = sigma + 2 * (int)(idx >> pl.w);
        const float* q = set.qn + (size_t)o * W;
        float* win = wins + (size_t)o * pl.Wp;
        const float qv = __ldg(q + k);
        const float qnext = k + 1 < W ? __ldg(q + k + 1) : 0.0f;
        win[4 + k] = map_into(lo_c, d_c, hi_c, qv);
        const bool pass = map_into(lo_l, d_l, hi_l, qv) <= L;
        const bool pass_next = k + 1 < W && map_into(lo_l, d_l, hi_l, qnext) <= L;
        if (k == 0 && !pass) win[0] = __int_as_float(0);
        if (pass && !pass_next) win[0] = __int_as_float(k + 1);
      }
    }
  }
  if (early) pdl_wait();  // thresholds and rows come from k_solve

  const size_t ps = (size_t)p * 2 + sigma;
  const float* th_g = set.theta + ps * d.theta_cap;
  // this candidate's row of the base solve's row table (word k at k K4), when
  // the solve built one; with at most one threshold per thread and a table
  // that holds every threshold the model allows, each thread loads its
  // threshold and word together with the count (one memory round trip; the
  // entries past the count are never used)
  const int* rt_g = set.rtab ? set.rtab + ps * kRowTabMax + rr : nullptr;
  const bool ahead = d.theta_cap <= (int)blockDim.x && d.K4 * d.theta_cap <= kRowTabMax;
  float th_a = 0.0f;
  int rt_a = 0;
  if (ahead && tid < d.theta_cap) {
    th_a = th_g[tid];
    if (rt_g) rt_a = rt_g[(size_t)tid * d.K4];
  }
  // a count above the launch's bound (reported below; the call then fails) is
  // cut to it, so that no index passes the shared arrays
  const int total_raw = set.ntheta[ps];
  const int total = min(total_raw, th_cap);
  const bool rtab = rt_g != nullptr && d.K4 * total <= kRowTabMax;
  int* sRt = reinterpret_cast<int*>(sTh + th_cap);  // [min(th_cap, kRowTabMax / 4)]
  for (int rho = tid; rho < d.K4; rho += blockDim.x) sC[rho] = set.rowC[ps * d.K4 + rho];
  if (ahead) {
    if (tid < total) {
      sTh[tid] = th_a;
      if (rtab) sRt[tid] = rt_a;  // (the words' shared array exists only with a table)
    }
  } else {
    for (int k = tid; k < total; k += blockDim.x) {
      sTh[k] = th_g[k];
      if (rtab) sRt[k] = rt_g[(size_t)k * d.K4];
    }
  }
  __syncthreads();
  if (total_raw > th_cap && tid == 0) atomicOr(set.status, ST_TABLE);
  const float cx = s_cx, cmax = s_cmax;
  const int msent = d.K == 1 ? rep_cap(d, jr) : 0;  // above every threshold only a lone class can go on

  // b0: last index feasible at Cexcl; b1: last index feasible at max(Cexcl, cap_hi).
  // Feasibility is nonincreasing along the sorted thresholds, so with the row
  // table each is the count of feasible indices less one (one barrier per 256
  // indices); without it, a joint search.
  int b0, b1;
  if (rtab) {
    int n0 = 0, n1 = 0;
    for (int k0 = 0; k0 < total; k0 += blockDim.x) {
      const int k = k0 + tid;
      bool f0 = false, f1 = false;
      if (k < total) {
        const int e = sRt[k], m = e & 0xFFFF;
        const bool other = (e >> 16) & 1;
        const float te = FL ? fmaxf(sTh[k], dle) : sTh[k];
        f0 = other || (m >= 1 && fulfil_r((float)m, cx, lam, rl) >= te);
        f1 = other || (m >= 1 && fulfil_r((float)m, cmax, lam, rl) >= te);
      }
      n0 += __syncthreads_count(f0);
      n1 += __syncthreads_count(f1);
    }
    b0 = n0 - 1;
    b1 = n1 - 1;
  } else {
    // Joint search: each round every group of gsz lanes probes one index and
    // answers for both capacities; each warp merges the answers with integer
    // max / min reductions, so a round costs one barrier.
    int lgs = 2;
    while ((1 << lgs) < d.K4 && lgs < 5) ++lgs;
    const int gsz = 1 << lgs, ng = (int)blockDim.x >> lgs, g = tid >> lgs, gl = tid & (gsz - 1);
    int lo0 = -1, hi0 = total, lo1 = -1, hi1 = total;
    for (int par = 0; hi0 - lo0 > 1 || hi1 - lo1 > 1; par ^= 1) {
      const int k = probe_index(g, ng, lo0, hi0, lo1, hi1);
      const float t = sTh[k];
      const Eval e = group_eval_excl<FL>(t, sC, sLam, sRl, sDl, d, rr, ie, gl, gsz);
      if (gl == 0) {
        const int m = replicas_left(e, jr, d);
        const float te = FL ? fmaxf(t, dle) : t;
        const int f = (feasible_at(e, m, cx, te, lam, rl) ? 1 : 0) | (feasible_at(e, m, cmax, te, lam, rl) ? 2 : 0);
        s_res[par][g] = k | (f << 24);
      }
      __syncthreads();
      int a0 = lo0, c0 = hi0, a1 = lo1, c1 = hi1;
      if (lane < ng) {
        const int v = s_res[par][lane];
        const int kq = v & 0xFFFFFF, f = v >> 24;
        if (f & 1) a0 = max(a0, kq); else c0 = min(c0, kq);
        if (f & 2) a1 = max(a1, kq); else c1 = min(c1, kq);
      }
      lo0 = __reduce_max_sync(0xffffffffu, a0);
      hi0 = __reduce_min_sync(0xffffffffu, c0);
      lo1 = __reduce_max_sync(0xffffffffu, a1);
      hi1 = __reduce_min_sync(0xffffffffu, c1);
    }
    b0 = lo0;
    b1 = lo1;
  }
  const int Lt = b1 - b0;
  // Three arrays of Lpad = max(P, 4) entries, P = pow2 >= Lt + 1 (at least 4
  // for 16-byte copies): kappa[u] for u < Lt, +inf beyond, so the scenario
  // search needs no bound checks; thx[pos] = the threshold reached with pos
  // kappa entries passed (thx[0] = theta_b0, 0 if b0 = -1) and mnx[pos] =
  // the replicas row r may use just above it, for pos = 0..Lt.
  int P = 1;
  while (P < Lt + 1) P <<= 1;
  const int Lpad = max(P, 4);
  if (Lpad > d.lcap) {  // cannot happen: Lt <= total <= theta_cap
    if (tid == 0) atomicOr(set.status, ST_TABLE);
    return;
  }
  float* kap = tab + kTableHeader;
  float* thx = kap + Lpad;
  float* mnx = thx + Lpad;

  // u = 0..Lt: m at index b0+1+u; kappa for u < Lt
  if (rtab) {
    // one thread per entry, m from the row table, kappa by a walk from the
    // estimate t lambda / m (Cexcl = -0 as +0: the same smallest capacity)
    const uint32_t bx = __float_as_uint(cx) & 0x7fffffffu, bmax = __float_as_uint(cmax) & 0x7fffffffu;
    for (int u = tid; u <= Lt; u += blockDim.x) {
      const int k = b0 + 1 + u;
      const int m = k < total ? (sRt[k] & 0xFFFF) : msent;
      if (u < Lt) {
        const float th = sTh[k], t = FL ? fmaxf(th, dle) : th;
        const float c0 = __fdividef(__fmul_rn(t, lam), (float)m);  // an estimate: the walk is exact
        kap[u] = __uint_as_float(kappa_walk((float)m, t, lam, rl, bx, bmax, __float_as_uint(c0)));
        thx[u + 1] = th;
      }
      if (m >= 1) s_row = 1;
      mnx[u] = (float)m;
    }
  } else {
    for (int u = warp; u <= Lt; u += nwarp) {
      const int k = b0 + 1 + u;
      int m;
      if (k < total) {
        const Eval e = group_eval_excl<FL>(sTh[k], sC, sLam, sRl, sDl, d, rr, ie, lane, 32);
        m = replicas_left(e, jr, d);
      } else {
        m = msent;
      }
      if (u < Lt) {
        // smallest capacity in (cx, cmax] at which f(m, C) >= max(theta_k,
        // delta_{i_e}), on the bit patterns of nonnegative floats (ordered like
        // the values). First the 32 patterns around the real solution t lambda / m,
        // one per lane; if the answer is not among them, a 32-ary search over the
        // whole interval.
        const float th = sTh[k], t = FL ? fmaxf(th, dle) : th;
        // Cexcl = -0 as +0 (the same smallest capacity), as in the table branch
        const uint32_t bx = __float_as_uint(cx) & 0x7fffffffu, bmax = __float_as_uint(cmax) & 0x7fffffffu;
        const float c0 = __fdividef(__fmul_rn(t, lam), (float)m);  // an estimate: the window is checked exactly
        const long long pl_ = (long long)__float_as_uint(c0) - 16 + lane;
        const uint32_t pt0 = pl_ < 0 ? 0u : (uint32_t)pl_;
        const bool ok0 = pt0 > bx && (pt0 >= bmax || fulfil_r((float)m, __uint_as_float(pt0), lam, rl) >= t);
        const uint32_t bal0 = __ballot_sync(0xffffffffu, ok0);
        uint32_t lo = bx, hi = bmax;
        if (bal0 != 0u && (bal0 & 1u) == 0u) {  // lane 0 fails, some lane passes: the first passing lane
          hi = __shfl_sync(0xffffffffu, pt0, __ffs(bal0) - 1);
          lo = hi - 1;
        }
        while (hi - lo > 1) {
          const uint32_t span = hi - lo;
          const uint32_t pt = lo + (uint32_t)(((uint64_t)(lane + 1) * span) >> 5);
          const bool ok = fulfil_r((float)m, __uint_as_float(pt), lam, rl) >= t;
          const uint32_t bal = __ballot_sync(0xffffffffu, ok);
          const int l = __ffs(bal) - 1;  // lane 31 tests hi, which is feasible
          const uint32_t nhi = __shfl_sync(0xffffffffu, pt, l);
          const uint32_t nlo = __shfl_sync(0xffffffffu, pt, l > 0 ? l - 1 : 0);
          if (l > 0) lo = nlo;
          hi = nhi;
        }
        if (lane == 0) {
          kap[u] = __uint_as_float(hi);
          thx[u + 1] = th;
        }
      }
      if (lane == 0) {
        if (m >= 1) s_row = 1;
        mnx[u] = (float)m;
        }
    }
  }
  for (int u = Lt + tid; u < Lpad; u += blockDim.x) {
    kap[u] = __int_as_float(0x7f800000);
    if (u > Lt) {
      thx[u] = 0.0f;
      mnx[u] = 0.0f;
    }
  }
  if (tid == 0) thx[0] = b0 >= 0 ? sTh[b0] : 0.0f;
  __syncthreads();
  if (tid == 0) {
    // every row-term quotient x / lambda of a scenario has x = m C' with
    // 1 <= m <= 32767 and C' in {0} or [min(Cexcl, cap_lo), cmax]: in
    // Markstein's range unless a positive C' can fall below 2^-60
    // (under the prior every C' lies in [cx, cmax])
    const bool fast = in_markstein_range(lam) && cmax <= 0x1p44f &&
                      (cx >= 0x1p-60f || (!RF && cx == 0.0f && (lo_c >= 0x1p-60f || hi_c == 0.0f)));
    tab[H_TH_BASE] = b0 >= 0 ? sTh[b0] : 0.0f;
    // t* at row capacity Cexcl (no kappa entry is at or below it): the value of
    // every scenario of this candidate whose tail gate is closed
    tab[H_TCL] = tstar_of<2, FL>(cx, kap, thx, mnx, Lt ? P >> 1 : 0, lam, rl, dle);
    tab[H_L] = __int_as_float(Lt);
    tab[H_LPAD] = __int_as_float(Lpad);
    tab[H_CX] = s_pc;
    tab[H_BX] = __int_as_float(s_bx);
    tab[H_PO] = s_po;
    tab[H_LAM] = lam;
    tab[H_LF] = s_lf;
    tab[H_HF] = s_hf;
    tab[H_LO_L] = lo_l;
    tab[H_HI_L] = hi_l;
    tab[H_SLO] = L;
    tab[H_CELL] = __int_as_float(cell);
    tab[H_P] = __int_as_float(p);
    tab[H_STEP0] = __int_as_float(Lt ? P >> 1 : 0);
    tab[H_ROW] = __int_as_float(s_row);
    tab[H_FAST] = __int_as_float(fast ? 1 : 0);
    tab[H_RLAM] = rl;
    tab[H_DLT] = dle;
  }
  // k_score launches only now: its blocks, resident early, slowed the base
  // solve and this kernel more than their early start saved
  pdl_trigger();
}

// t* of one realisation with row capacity C (see the file comment). kap is
// padded with +inf to a power of two above the entry count, so the
// branch-free search needs no bound checks; step0 = half that power. thx[pos]
// and mnx[pos] are the threshold and the replicas of row r once pos entries
// are passed. ROW = 0: no reachable threshold leaves row r a replica (m < 1
// throughout), so the row term is 0; ROW = 1: the quotient by Markstein's
// method (valid for every C' of the segment); ROW = 2: the IEEE division.
// FL: the candidate's class is critical and row r's term counts only at or
// above its floor dl.
template <int ROW, bool FL>
__device__ __forceinline__ float tstar_of(float C, const float* kap, const float* thx, const float* mnx,
                                          int step0, float lam, float rlam, float dl) {
  int pos = 0;
  for (int step = step0; step > 0; step >>= 1) pos += kap[pos + step - 1] <= C ? step : 0;
  const float thb = thx[pos];
  if (ROW == 0) return thb;
  const float m = mnx[pos];
  float tr;
  if (ROW == 1) tr = m >= 1.0f ? fulfil_fast(m, C, lam, rlam) : 0.0f;
  else tr = m >= 1.0f ? fulfil(m, C, lam) : 0.0f;
  if (FL) return (tr > thb && tr >= dl) ? tr : thb;
  return tr > thb ? tr : thb;
}

// Sum of rint(g 2^40) over values 0 <= g <= 1 (every Gamma' is in [0, 1]).
// u = RN(g + 8) - 8 is g rounded to the 2^-20 grid (the spacing of floats in
// [8, 16)) and exact, and d = g - u is exact with |d| <= 2^-21, so
// rint(g 2^40) = u 2^40 + rint(d 2^40) (u 2^40 is an even integer). The two
// terms are the bit patterns of 2^23 + u 2^20 and 1.5 2^23 + d 2^40 less the
// patterns of 2^23 and 1.5 2^23 (one FMA each; the second rounds d 2^40 to an
// integer, ties to even); they are summed in two 32-bit words and the offsets
// removed once: exact for up to 2048 values, with adds and FMAs only.
struct Acc40 {
  uint32_t h = 0, l = 0, n = 0;
  __device__ __forceinline__ void add(float g) {
    const float u = __fsub_rn(__fadd_rn(g, 8.0f), 8.0f);
    const float dl = __fsub_rn(g, u);
    h += __float_as_uint(__fmaf_rn(u, 0x1p20f, 0x1p23f));
    l += __float_as_uint(__fmaf_rn(dl, 0x1p40f, 0x1.8p23f));
  }
  __device__ __forceinline__ uint64_t value() const {
    const uint32_t H = h - n * 0x4B000000u;
    const int32_t Lo = (int32_t)(l - n * 0x4B400000u);
    return ((uint64_t)H << 20) + (uint64_t)(int64_t)Lo;
  }
};

// Cheapest cover of threshold t by class i in one scenario (dump mode only):
// rows from the base realisation except row rr, which has capacity C and bin
// bC. Returns the cost (kCostInf: none) and the choice code.
__device__ int dump_cover(float t, const Set& set, size_t ps, int rr, float C, int bC, int i, uint32_t* code) {
  const Dims& d = set.d;
  int best = kCostInf, bj = -1, bn = 0, bbin = -1;
  for (int j = 0; j < kT; ++j) {
    const int rho = 4 * i + j;
    const float c = rho == rr ? C : set.rowC[ps * d.K4 + rho];
    const int b = rho == rr ? bC : set.rowB[ps * d.K4 + rho];
    if (b < 0) continue;
    const int n = min_replicas(t, c, set.lam[i], __frcp_rn(set.lam[i]), rep_capf(d, j));
    if (n && (n << j) < best) {
      best = n << j;
      bj = j;
      bn = n;
      bbin = b;
    }
  }
  *code = bj >= 0 ? ((uint32_t)bn | ((uint32_t)bj << 16) | ((uint32_t)bbin << 18)) : 0u;
  return best;
}

// Per-class choice of one scenario at threshold t (dump mode only): the cover
// of max(t, delta_i) when t > 0; with t = 0, the critical classes' floor
// covers when they fit in G together, else nothing.
template <bool FL>
__device__ void dump_choices(float t, const Set& set, size_t ps, int rr, float C, int bC,
                             uint32_t* choice, int32_t* total_gpus) {
  const Dims& d = set.d;
  int total = 0;
  if (t > 0.0f) {
    for (int i = 0; i < d.K; ++i) {
      const float dl = FL ? set.slo[d.K + i] : 0.0f;
      const int c = dump_cover(fmaxf(t, dl), set, ps, rr, C, bC, i, &choice[i]);
      if (c < kCostInf) total += c;
    }
  } else {
    bool met = true;
    for (int i = 0; i < d.K; ++i) {
      const float dl = FL ? set.slo[d.K + i] : 0.0f;
      choice[i] = 0u;
      if (dl > 0.0f) {
        const int c = dump_cover(dl, set, ps, rr, C, bC, i, &choice[i]);
        if (c < kCostInf) total += c; else met = false;
      }
    }
    if (!met || total > d.G) {
      total = 0;
      for (int i = 0; i < d.K; ++i) choice[i] = 0u;
    }
  }
  *total_gpus = total;
}

// Philox calls [q_lo, q_hi) of one (candidate, outcome) segment; call q
// serves samples 4q..4q+3, sample 4q+h reading output word h (upper 16 bits:
// capacity position, lower 16 bits: tail position; top w = log2(W) bits
// each). win is the staged window of the outcome (gate position, then the
// mapped capacities); h0/h1 point at the staged table headers; kap/thx/mnx at
// the table arrays (shared memory when TS, else global). The capacity
// position is floor(word W / 2^32) (the top w bits); the tail gate of Eq. 5
// (l_y <= L_i), a position test kl < kgate, is the lower half compared with
// kgate << (16 - w). With capacities >= 0, max(Cexcl, gate ? c_y : 0) is the
// patched row capacity.
struct PieceSum {
  Acc40 acc;       // the last at most 1024 values
  uint64_t total;  // earlier values, flushed
};

template <bool TS, int ROW, bool FL, bool RF>
__device__ __forceinline__ PieceSum run_piece(const Plan& pl, const PhiloxKeys& keys, int o, int q_lo, int q_hi,
                                              const float* win, const float* h0, const float* h1,
                                              const float* kap0, const float* thx0, const float* mnx0,
                                              const float* kap1, const float* thx1, const float* mnx1) {
  const int st0 = __float_as_int(h0[H_STEP0]), st1 = __float_as_int(h1[H_STEP0]);
  const float cx0 = h0[H_CX], cx1 = h1[H_CX];
  const RowCap rc0 = row_cap_of(h0), rc1 = row_cap_of(h1);
  const float lam = h0[H_LAM], rlam = h0[H_RLAM], dl = h0[H_DLT];
  const int cell = __float_as_int(h0[H_CELL]);
  const uint32_t ctr1 = (uint32_t)o, ctr2 = (uint32_t)cell, ctr3 = pl.round;
  const uint32_t w = (uint32_t)pl.w;  // W = 2^w positions
  const uint32_t kgs = (uint32_t)__float_as_int(win[0]) << pl.sh;
  const float* sQo = win + 4;
  Acc40 acc;
  uint64_t total = 0;
  auto eval = [&](uint32_t word) {
    const float cy = sQo[__funnelshift_lc(word, 0u, w)];  // floor(word W / 2^32)
    const bool g = (word & 0xFFFFu) < kgs;
    const float cyg = g ? cy : 0.0f;
    const float c0 = RF ? row_cap(rc0, cy, g) : fmaxf(cx0, cyg);
    const float c1 = RF ? row_cap(rc1, cy, g) : fmaxf(cx1, cyg);
    const float t0 = tstar_of<ROW, FL>(c0, kap0, thx0, mnx0, st0, lam, rlam, dl);
    const float t1 = tstar_of<ROW, FL>(c1, kap1, thx1, mnx1, st1, lam, rlam, dl);
    acc.add(__fsub_rn(t1, t0));
  };
  const int q_full = min(q_hi, pl.S >> 2);  // calls whose four samples all exist
  const int step = (int)blockDim.x;
  int q = q_lo + (int)threadIdx.x;
  while (q < q_full) {
    // at most 256 calls (1024 values) between flushes of the 32-bit sums
    const int q_end = min(q_full, q + 256 * step);
    for (; q < q_end; q += step) {
      const uint4 x = philox4x32_10(make_uint4((uint32_t)q, ctr1, ctr2, ctr3), keys);
      eval(x.x);
      eval(x.y);
      eval(x.z);
      eval(x.w);
      acc.n += 4;
    }
    if (q < q_full) {
      total += acc.value();
      acc = Acc40();
    }
  }
  if (q < q_hi) {  // the segment's last call, serving S mod 4 samples
    const uint4 x = philox4x32_10(make_uint4((uint32_t)q, ctr1, ctr2, ctr3), keys);
    const int nv = pl.S - 4 * q;
    eval(x.x);
    if (nv > 1) eval(x.y);
    if (nv > 2) eval(x.z);
    acc.n += (uint32_t)nv;
  }
  return PieceSum{acc, total};
}

// The same calls in dump mode: every scenario also writes its record (draws,
// both t* and the per-class choices), with l_y mapped from the raw quantile
// and the gate compared with the SLO directly.
// Bin of row r's capacity in one scenario under the monotone prior (dump mode
// only): the refit row's SLO-feasible bins in realisation sg, the largest
// capacity, ties to the lower bin; -1 when none.
__device__ int refit_bin(const Set& set, int p, int sg, int rr, int be, float cy, float ly, float L) {
  const Dims& d = set.d;
  const float* bp = set.bounds + (size_t)p * 4 * d.cells + (size_t)rr * d.B;
  const float* cl = bp + (size_t)CAP_LO * d.cells;
  const float* ch = bp + (size_t)CAP_HI * d.cells;
  const float* tl = bp + (size_t)TAIL_LO * d.cells;
  const float* th = bp + (size_t)TAIL_HI * d.cells;
  float best = 0.0f;
  int bb = -1;
  for (int b = 0; b < d.B; ++b) {
    float c, t;
    if (b == be) {
      c = cy;
      t = ly;
    } else if (b > be) {  // higher load: lower bounds rise to the draw
      c = sg ? ch[b] : raise_lo(cl[b], ch[b], cy);
      t = sg ? raise_lo(tl[b], th[b], ly) : th[b];
    } else {              // lower load: upper bounds fall to the draw
      c = sg ? lower_hi(cl[b], ch[b], cy) : cl[b];
      t = sg ? tl[b] : lower_hi(tl[b], th[b], ly);
    }
    if (t <= L && (bb < 0 || c > best)) {
      best = c;
      bb = b;
    }
  }
  return bb;
}

template <bool TS, bool FL, bool RF>
__device__ uint64_t run_piece_dump(const Set& set, const Plan& pl, int item, int o, int q_lo, int q_hi,
                                   const float* win, const float* h0, const float* h1, const float* kap0,
                                   const float* thx0, const float* mnx0, const float* kap1, const float* thx1,
                                   const float* mnx1, unsigned char* dump, int dump_stride) {
  const int st0 = __float_as_int(h0[H_STEP0]), st1 = __float_as_int(h1[H_STEP0]);
  const float cx0 = h0[H_CX], cx1 = h1[H_CX];
  const RowCap rc0 = row_cap_of(h0), rc1 = row_cap_of(h1);
  const float lam = h0[H_LAM], rlam = __frcp_rn(lam), dl = h0[H_DLT];
  const int cell = __float_as_int(h0[H_CELL]), p = __float_as_int(h0[H_P]);
  const PhiloxKeys keys = philox_keys(pl.key0, pl.key1 ^ (pl.stream_base + (uint32_t)p));
  const uint32_t sh = (uint32_t)pl.sh;
  const int S = pl.S;
  const uint32_t ctr1 = (uint32_t)o, ctr2 = (uint32_t)cell, ctr3 = pl.round;
  const float* sQo = win + 4;
  const float lo_l = h0[H_LO_L], hi_l = h0[H_HI_L];
  uint64_t acc = 0;
  for (int q = q_lo + (int)threadIdx.x; q < q_hi; q += blockDim.x) {
    const uint4 x = philox4x32_10(make_uint4((uint32_t)q, ctr1, ctr2, ctr3), keys);
    for (int h = 0; h < 4; ++h) {
      const int s = 4 * q + h;
      if (s >= S) break;  // the last call may serve fewer than four samples
      const uint32_t word = h == 0 ? x.x : h == 1 ? x.y : h == 2 ? x.z : x.w;
      const int kc = (int)((word >> 16) >> sh);
      const int kl = (int)((word & 0xFFFFu) >> sh);
      const float cy = sQo[kc];
      const float ly = map_into(lo_l, __fsub_rn(hi_l, lo_l), hi_l, set.qn[(size_t)o * pl.W + kl]);
      const bool gate = ly <= h0[H_SLO];
      const float C0 = RF ? row_cap(rc0, cy, gate) : gate ? fmaxf(cx0, cy) : cx0;
      const float C1 = RF ? row_cap(rc1, cy, gate) : gate ? fmaxf(cx1, cy) : cx1;
      const float t0 = tstar_of<2, true>(C0, kap0, thx0, mnx0, st0, lam, rlam, dl);
      const float t1 = tstar_of<2, true>(C1, kap1, thx1, mnx1, st1, lam, rlam, dl);
      acc += fixed40(__fsub_rn(t1, t0));
      const size_t idx = ((size_t)item * pl.O + o) * pl.S + s;
      unsigned char* rec = dump + idx * dump_stride;
      fs_scenario_head hd;
      hd.c_y = cy;
      hd.l_y = ly;
      hd.t_star[0] = t0;
      hd.t_star[1] = t1;
      const int rr = cell / set.d.B, be = cell - rr * set.d.B;
      uint32_t* ch = reinterpret_cast<uint32_t*>(rec + sizeof(fs_scenario_head));
      for (int sg = 0; sg < 2; ++sg) {
        const float cx = sg ? cx1 : cx0;
        const int bx = __float_as_int(sg ? h1[H_BX] : h0[H_BX]);
        int bC;
        if (RF) bC = refit_bin(set, p, sg, rr, be, cy, ly, h0[H_SLO]);
        else if (!gate) bC = bx;
        else if (bx < 0 || cy > cx) bC = be;
        else if (cy == cx) bC = min(be, bx);
        else bC = bx;
        dump_choices<FL>(sg ? t1 : t0, set, (size_t)p * 2 + sg, rr, sg ? C1 : C0, bC, ch + sg * set.d.K,
                     &hd.total_gpus[sg]);
      }
      *reinterpret_cast<fs_scenario_head*>(rec) = hd;
    }
  }
  return acc;
}

// Table path. Within a segment (candidate e, outcome o) a scenario's Gamma'
// depends on its draw only through the capacity position k (which selects c_y
// among the outcome's W mapped quantiles) and the tail gate (l_y <= L_i); with
// the gate closed the row keeps Cexcl whatever k is. So the segment has at most
// W + 1 values of rint(Gamma' 2^40): gtab[k] for an open gate at position k,
// gtab[W] for a closed gate. The closed-gate value comes from the two t* at
// Cexcl that the preparation stored (H_TCL); the block evaluates the W others
// once per chunk (two t* each, the same arithmetic as a scenario), after which
// a scenario costs its share of the Philox call, one index and one
// shared-memory load. Each entry is the value as one 64-bit word.
// Without the prior an entry whose capacity is at or below a realisation's
// Cexcl leaves that row at Cexcl, so its t* is the closed-gate one (H_TCL)
// and is not evaluated again.
// RF: under the monotone prior the closed-gate values also depend on the
// position (the draw refits the row's other bins): entries [W, 2W) hold them,
// evaluated when `closed` (the open half when `open`).
// Returns the number of t* this thread evaluated (the measurement's count).
template <bool TS, int ROW, bool FL, bool RF>
__device__ __forceinline__ int build_gtab(uint64_t* gtab, int W, const float* win, const float* h0, const float* h1,
                                           const float* kap0, const float* thx0, const float* mnx0,
                                           const float* kap1, const float* thx1, const float* mnx1,
                                           bool open = true, bool closed = false) {
  const int st0 = __float_as_int(h0[H_STEP0]), st1 = __float_as_int(h1[H_STEP0]);
  const float cx0 = h0[H_CX], cx1 = h1[H_CX];
  const float tcl0 = h0[H_TCL], tcl1 = h1[H_TCL];
  const RowCap rc0 = row_cap_of(h0), rc1 = row_cap_of(h1);
  const float lam = h0[H_LAM], rlam = h0[H_RLAM], dl = h0[H_DLT];
  const float* capw = win + 4;
  const int k0 = (RF && !open) ? W : 0, k1 = (RF && closed) ? 2 * W : W;
  int evals = 0;
  for (int k = k0 + (int)threadIdx.x; k < k1; k += blockDim.x) {
    const bool g = k < W;
    const float cy = capw[g ? k : k - W];
    const float c0 = RF ? row_cap(rc0, cy, g) : fmaxf(cx0, cy);
    const float c1 = RF ? row_cap(rc1, cy, g) : fmaxf(cx1, cy);
    // at or below Cexcl the row keeps Cexcl: t* is the closed-gate one
    const bool e0 = RF || cy > cx0, e1 = RF || cy > cx1;
    const float t0 = e0 ? tstar_of<ROW, FL>(c0, kap0, thx0, mnx0, st0, lam, rlam, dl) : tcl0;
    const float t1 = e1 ? tstar_of<ROW, FL>(c1, kap1, thx1, mnx1, st1, lam, rlam, dl) : tcl1;
    evals += (int)e0 + (int)e1;
    const uint64_t gv = fixed40(__fsub_rn(t1, t0));
    gtab[k] = gv;
  }
  return evals;
}

// Work decomposition of one k_score launch: segment = (item, outcome) with
// pl.calls Philox calls; a chunk is up to `chunk` consecutive calls of one
// segment, nch chunks per segment.
struct ScoreGrid {
  int total;        // chunks (< 2^31: the host widens chunks until they fit)
  int chunk;        // calls per chunk (a multiple of the block size)
  int nch;          // chunks per segment
  int lcap_s;       // table entries staged per realisation
  int tcopy;        // floats staged per table: header + 3 lcap_s
  int dyn;          // 1: chunks after the first two come from the counter; 0: chunk b + k gridDim
};

// Which scoring path a launch takes.
enum : int { SCORE_PLAIN = 0, SCORE_DUMP = 1, SCORE_TABLE = 2, SCORE_TABLE_MULTI = 3 };

// Thread 0: stage the data of segment seg (its outcome window and both
// candidate tables, header plus lcap_s entries each) into dst, completing on bar.
__device__ __forceinline__ void stage_segment(const Set& set, const Plan& pl, const float* rec, int seg,
                                              float* dst, uint64_t* bar, int tcopy) {
  const int item = seg >> pl.logO, o = seg & (pl.O - 1);
  const float* r = rec + (size_t)item * pl.item_floats;
  const uint32_t tb = (uint32_t)tcopy * 4u, wb = (uint32_t)pl.Wp * 4u;
  fence_proxy_async();
  mbar_expect_tx(bar, wb + 2 * tb);
  bulk_g2s(dst, r + 2 * (size_t)set.d.slot_floats + (size_t)o * pl.Wp, wb, bar);
  bulk_g2s(dst + pl.Wp, r, tb, bar);
  bulk_g2s(dst + pl.Wp + tcopy, r + set.d.slot_floats, tb, bar);
}

// Blocks take chunks until none is left: chunk blockIdx.x, then chunk
// blockIdx.x + gridDim.x, then (with many chunks per block) chunks handed out
// by a global counter, so segments of unequal cost (table length, row-term
// divisions) even out across the SMs; with few chunks per block the
// assignment stays static (every block would meet the counter at once). A chunk's data are staged in shared memory by TMA bulk copies,
// double-buffered: thread 0 issues the next chunk's copies (and the counter
// increment whose result names the chunk after it) before this chunk is
// computed. The sums are integers, so the order of the chunks does not
// change the result.
// FL: some class is critical (the model has floors): row terms are gated by the
// candidate class's floor (0, so always passed, for a class that is not).
// GT: the table path (build_gtab), chosen by the host when a chunk's samples
// outnumber a segment's W + 1 table entries; never with DUMP. KC (table path,
// one problem): Philox round keys from the plan's parameters.
template <bool DUMP, bool FL, bool GT, bool KC, bool RF>
__global__ void __launch_bounds__(kScoreThreads, 4) k_score(Set set, Items it, Plan pl, const float* rec,
                                                         uint64_t* sums, unsigned char* dump, int dump_stride,
                                                         ScoreGrid sg) {
  extern __shared__ __align__(16) unsigned char smraw[];
  uint64_t* bar = reinterpret_cast<uint64_t*>(smraw);  // [2]
  float* stage0 = reinterpret_cast<float*>(smraw + 16);
  const int stage_floats = pl.Wp + 2 * sg.tcopy;
  // GT: two tables of W + 1 entries (2W under the prior), used by alternate
  // chunks; over several problems (short segments, blocks of 64 threads whose
  // count per SM shared memory limits) one table and one more barrier a chunk
  constexpr bool kOneTable = GT && !KC;
  uint64_t* gtab2 = reinterpret_cast<uint64_t*>(smraw + 16 + (size_t)2 * stage_floats * 4);
  const int gt_len = RF ? 2 * pl.W : pl.W + 1;
  // per stage: chunk index, its segment and its part (thread 0 divides once)
  __shared__ int s_chunk[2], s_seg[2], s_part[2];
  const Dims& d = set.d;  // kernel-parameter space: no local copy
  const int tid = threadIdx.x, lane = tid & 31;
  (void)it;

  pdl_wait();  // records, zeroed sums and the zeroed counter come from k_prep
  // the reduction kernel may be placed now: it waits for this grid to complete
  // before it reads anything
  pdl_trigger();
  const int g = (int)gridDim.x;
  int next = 0;  // thread 0: the chunk to stage next
  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    const int c0 = (int)blockIdx.x;  // the grid has at most sg.total blocks
    s_chunk[0] = c0;
    s_seg[0] = c0 / sg.nch;
    s_part[0] = c0 - s_seg[0] * sg.nch;
  }
  __syncthreads();
  if (tid == 0) {
    stage_segment(set, pl, rec, s_seg[0], stage0, &bar[0], sg.tcopy);
    next = (int)blockIdx.x + g;  // may pass sg.total: then the block stops after one chunk
  }
  // 32-bit warp sums are exact while a thread holds at most 32 values (the
  // table path splits its 64-bit sums: at most 128 values)
  const bool small = sg.chunk <= 8 * (int)blockDim.x;
  const bool small_gt = sg.chunk <= 32 * (int)blockDim.x;
  PhiloxKeys keys;
  int keys_p = -1;  // problem whose round keys are in `keys`

  for (int j = 0;; ++j) {
    const int st = j & 1;
    const int c = s_chunk[st];
    if (c >= sg.total) break;
    if (tid == 0) {
      s_chunk[st ^ 1] = next;
      if (next < sg.total) {
        const int sn = next / sg.nch;
        s_seg[st ^ 1] = sn;
        s_part[st ^ 1] = next - sn * sg.nch;
        stage_segment(set, pl, rec, sn, stage0 + (size_t)(st ^ 1) * stage_floats, &bar[st ^ 1], sg.tcopy);
        if (sg.dyn) {
          // consumed one chunk later; saturates at sg.total so that it cannot wrap
          const unsigned long long v = atomicAdd(set.work, 1ull) + 2ull * (unsigned long long)g;
          next = v < (unsigned long long)sg.total ? (int)v : sg.total;
        } else {
          next = (long long)next + g < (long long)sg.total ? next + g : sg.total;
        }
      }
    }
    // a thread whose wait succeeded may use the stage; the barrier at the end
    // of the chunk tells every thread whether any wait gave up
    const bool ok = mbar_wait(&bar[st], (uint32_t)((j >> 1) & 1), kWaitLimitNs);
    const float* stg = stage0 + (size_t)st * stage_floats;
    const float* h0 = stg + pl.Wp;
    const float* h1 = h0 + sg.tcopy;
    const int seg = s_seg[st], part = s_part[st];
    const int item = seg >> pl.logO, o = seg & (pl.O - 1);
    const int q_lo = part * sg.chunk;
    const int q_hi = min(q_lo + sg.chunk, pl.calls);
    if constexpr (GT) {
      // One barrier a chunk: every thread's reads of stage st (table build and
      // the gate position) come before it, so thread 0 may refill the stage
      // next iteration, and the next chunk builds the other table while a late
      // thread may still draw from this one (with one table, a second barrier
      // before the build).
      uint64_t* gtab = kOneTable ? gtab2 : gtab2 + (size_t)(j & 1) * gt_len;
      if (kOneTable) __syncthreads();  // every thread has drawn from the previous chunk's table
      const int cell = ok ? __float_as_int(h0[H_CELL]) : -1;
      const bool use = cell >= 0 && cell < d.cells;  // a bad device-side id was flagged by k_prep
      // passing tail positions of the stratum, as the top bits of a 16-bit field
      const uint32_t kgs = use ? (uint32_t)__float_as_int(stg[0]) << pl.sh : 0u;
      const uint32_t kgs16 = (uint32_t)min((unsigned long long)kgs << 16, 0xFFFFFFFFull);
      if (use) {
        const uint64_t gc = fixed40(__fsub_rn(h1[H_TCL], h0[H_TCL]));
        // under the prior: the halves the stratum's gate positions can reach
        const bool any_open = kgs != 0u, any_closed = kgs16 != 0xFFFFFFFFu;
        if (!RF && kgs == 0u) {
          // the gate is closed at every position of the stratum: every entry
          // is the closed-gate value, stored once at W (each scenario still
          // draws its position and loads its entry, with stride 0)
          if (tid == 0) gtab[pl.W] = gc;
        } else {
          if (tid == 0) {
            if (!RF) gtab[pl.W] = gc;
            // scenarios that test their tail gate (a stratum on both sides of the SLO)
            if (KC && part == 0 && any_open && any_closed) atomicAdd(&set.work[3], (unsigned long long)pl.S);
          }
          const int Lp0 = __float_as_int(h0[H_LPAD]), Lp1 = __float_as_int(h1[H_LPAD]);
          const bool r0 = __float_as_int(h0[H_ROW]) != 0, r1 = __float_as_int(h1[H_ROW]) != 0;
          const bool f0 = __float_as_int(h0[H_FAST]) != 0, f1 = __float_as_int(h1[H_FAST]) != 0;
          const int row = (!r0 && !r1) ? 0 : ((!r0 || f0) && (!r1 || f1)) ? 1 : 2;
          int evals;
#define FS_BUILD(TSV, ROWV, FLV)                                                                          \
  evals = build_gtab<TSV, ROWV, FLV, RF>(gtab, pl.W, stg, h0, h1, k0, k0 + Lp0, k0 + 2 * Lp0, k1, k1 + Lp1, \
                                         k1 + 2 * Lp1, any_open, any_closed)
#define FS_BUILDS(TSV)                       \
  if (row == 0) FS_BUILD(TSV, 0, false);     \
  else if (row == 1) FS_BUILD(TSV, 1, FL);   \
  else FS_BUILD(TSV, 2, FL);
          if (Lp0 <= sg.lcap_s && Lp1 <= sg.lcap_s) {
            const float* k0 = h0 + kTableHeader;
            const float* k1 = h1 + kTableHeader;
            FS_BUILDS(true)
          } else {
            const float* k0 = rec + (size_t)item * pl.item_floats + kTableHeader;
            const float* k1 = k0 + d.slot_floats;
            FS_BUILDS(false)
          }
#undef FS_BUILDS
#undef FS_BUILD
          if (KC && part == 0) {
            // t* evaluated, once per segment (later chunks of a segment
            // rebuild the same table): the measurement's algorithmic count
            evals = __reduce_add_sync(0xffffffffu, evals);
            if (lane == 0 && evals) atomicAdd(&set.work[2], (unsigned long long)evals);
          }
        }
        if (!KC) {
          const int p = __float_as_int(h0[H_P]);
          if (p != keys_p) {
            keys = philox_keys(pl.key0, pl.key1 ^ (pl.stream_base + (uint32_t)p));
            keys_p = p;
          }
        }
      }
      if (__syncthreads_or(!ok)) {  // the table is complete; or some wait gave up
        if (tid == 0) atomicOr(set.status, ST_TIMEOUT);
        if (!ok) mbar_wait(&bar[st], (uint32_t)((j >> 1) & 1), kWaitLimitNs);
        if (s_chunk[st ^ 1] < sg.total) mbar_wait(&bar[st ^ 1], (uint32_t)(((j + 1) >> 1) & 1), kWaitLimitNs);
        return;
      }
      uint64_t gs = 0;
      if (use) {
        if (kgs == 0u || kgs16 == 0xFFFFFFFFu)  // the gate is the same at every position
          gs = sample_gtab<KC, RF, false>(pl, keys, o, cell, q_lo, q_hi,
                                          smem_u32(gtab) + (kgs == 0u ? 8u * (uint32_t)pl.W : 0u), 0u,
                                          (!RF && kgs == 0u) ? pl.uniform_stride : pl.entry_bytes);
        else
          gs = sample_gtab<KC, RF, true>(pl, keys, o, cell, q_lo, q_hi, smem_u32(gtab), kgs16);
      }
      uint64_t v;
      if (small_gt) {
        // at most 128 values per thread (each at most 2^40): the total's bits
        // above bit 21 are at most 2^26 and the low 21 bits below 2^21, so
        // each part's warp sum fits in 32 bits
        const uint32_t H = __reduce_add_sync(0xffffffffu, (uint32_t)(gs >> 21));
        const uint32_t Lo = __reduce_add_sync(0xffffffffu, (uint32_t)gs & 0x1FFFFFu);
        v = ((uint64_t)H << 21) + (uint64_t)Lo;
      } else {
        v = gs;
        for (int off = 16; off; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
      }
      if (lane == 0 && v) atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)seg]), (unsigned long long)v);
      continue;
    } else {
    PieceSum ps{Acc40(), 0ull};
    uint64_t acc_dump = 0;
    if (ok) {
      const int Lp0 = __float_as_int(h0[H_LPAD]), Lp1 = __float_as_int(h1[H_LPAD]);
      const int cell = __float_as_int(h0[H_CELL]);
      if (cell >= 0 && cell < d.cells) {  // a bad device-side id was flagged by k_prep
        const bool r0 = __float_as_int(h0[H_ROW]) != 0, r1 = __float_as_int(h1[H_ROW]) != 0;
        const bool f0 = __float_as_int(h0[H_FAST]) != 0, f1 = __float_as_int(h1[H_FAST]) != 0;
        const int row = (!r0 && !r1) ? 0 : ((!r0 || f0) && (!r1 || f1)) ? 1 : 2;
        const int p = __float_as_int(h0[H_P]);
        if (!DUMP && p != keys_p) {
          keys = philox_keys(pl.key0, pl.key1 ^ (pl.stream_base + (uint32_t)p));
          keys_p = p;
        }
        // the table pointers stay in one address space per branch (shared or global)
#define FS_PIECE(TSV, ROWV, FLV)                                                                      \
  run_piece<TSV, ROWV, FLV, RF>(pl, keys, o, q_lo, q_hi, stg, h0, h1, k0, k0 + Lp0, k0 + 2 * Lp0, k1, k1 + Lp1, \
                                k1 + 2 * Lp1)
#define FS_PIECES(TSV) \
  (row == 0 ? FS_PIECE(TSV, 0, false) : row == 1 ? FS_PIECE(TSV, 1, FL) : FS_PIECE(TSV, 2, FL))
#define FS_DUMP(TSV)                                                                                       \
  run_piece_dump<TSV, FL, RF>(set, pl, item, o, q_lo, q_hi, stg, h0, h1, k0, k0 + Lp0, k0 + 2 * Lp0, k1, k1 + Lp1, \
                              k1 + 2 * Lp1, dump, dump_stride)
        if (Lp0 <= sg.lcap_s && Lp1 <= sg.lcap_s) {
          const float* k0 = h0 + kTableHeader;
          const float* k1 = h1 + kTableHeader;
          if constexpr (DUMP) acc_dump = FS_DUMP(true);
          else ps = FS_PIECES(true);
        } else {
          const float* k0 = rec + (size_t)item * pl.item_floats + kTableHeader;
          const float* k1 = k0 + d.slot_floats;
          if constexpr (DUMP) acc_dump = FS_DUMP(false);
          else ps = FS_PIECES(false);
        }
#undef FS_DUMP
#undef FS_PIECES
#undef FS_PIECE
      }
    }
    if (!DUMP && small) {
      // at most 32 values per thread: each part's warp sum fits in 32 bits
      const uint32_t H = __reduce_add_sync(0xffffffffu, ps.acc.h - ps.acc.n * 0x4B000000u);
      const int32_t Lo = (int32_t)__reduce_add_sync(0xffffffffu, ps.acc.l - ps.acc.n * 0x4B400000u);
      const uint64_t v = ((uint64_t)H << 20) + (uint64_t)(int64_t)Lo;
      if (lane == 0 && v) atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)seg]), (unsigned long long)v);
    } else {
      uint64_t v = DUMP ? acc_dump : ps.total + ps.acc.value();
      for (int off = 16; off; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
      if (lane == 0 && v) atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)seg]), (unsigned long long)v);
    }
    }
    // stage st is free for the copies issued next iteration
    if (__syncthreads_or(!ok)) {
      if (tid == 0) atomicOr(set.status, ST_TIMEOUT);
      // let copies in flight land before the block exits (bounded as well)
      if (!ok) mbar_wait(&bar[st], (uint32_t)((j >> 1) & 1), kWaitLimitNs);
      if (s_chunk[st ^ 1] < sg.total) mbar_wait(&bar[st ^ 1], (uint32_t)(((j + 1) >> 1) & 1), kWaitLimitNs);
      return;
    }
  }
}

__global__ void k_finalize(Set set, Items it, Plan pl, const uint64_t* sums, double* gap, double* score,
                           float* gamma_t, int32_t* best, uint32_t* status_copy) {
  pdl_wait();
  const int p = blockIdx.x;
  const int beg = it.off ? it.off[p] : 0;
  const int end = it.off ? it.off[p + 1] : it.n;
  const Best b = finalize_problem(set, it, pl, sums, p, beg, end, gap, score, gamma_t ? gamma_t + p : nullptr, beg);
  if (threadIdx.x == 0 && best) best[p] = b.valid() ? b.cell : -1;
  // every kernel of the call has finished (stream order, and the wait above):
  // its status word can travel with the outputs
  if (threadIdx.x == 0 && p == 0 && status_copy) *status_copy = *set.status;
}

// One problem with many candidates, split over the CTAs: each writes its
// candidates' expectations and scores and its best entry into part[2 b ..],
// and the last to finish (a ticket in work[1], zeroed by k_prep) reduces them.
__global__ void k_finalize_split(Set set, Items it, Plan pl, const uint64_t* sums, double* gap, double* score,
                                 float* gamma_t, int32_t* best, uint32_t* status_copy, uint64_t* part) {
  pdl_wait();
  const int nb = (int)gridDim.x, per = (it.n + nb - 1) / nb;
  const int beg = min(it.n, (int)blockIdx.x * per), end = min(it.n, beg + per);
  const Best b = finalize_problem(set, it, pl, sums, 0, beg, end, gap, score,
                                  blockIdx.x == 0 ? gamma_t : nullptr, 0);
  __shared__ int s_last;
  if (threadIdx.x == 0) {
    part[2 * blockIdx.x] = (uint64_t)b.hi;
    part[2 * blockIdx.x + 1] = ((uint64_t)b.lo << 32) | (uint32_t)b.cell;
    __threadfence();
    s_last = atomicAdd(&set.work[1], 1ull) == (unsigned long long)(nb - 1);
  }
  __syncthreads();
  if (!s_last || threadIdx.x >= 32) return;
  __threadfence();
  Best r = no_best();
  for (int q = threadIdx.x; q < nb; q += 32) {
    const uint64_t w = __ldcg(part + 2 * q + 1);
    const Best c{(long long)__ldcg(part + 2 * q), (uint32_t)(w >> 32), (int)(uint32_t)w};
    if (better(c, r)) r = c;
  }
  r = warp_best(r);
  if (threadIdx.x == 0) {
    if (best) *best = r.valid() ? r.cell : -1;
    if (status_copy) *status_copy = *set.status;
  }
}

// rowC, the thresholds and, with a row table, the candidate row's words
static size_t prep_smem_bytes(const Set& set, int th_cap) {
  return (size_t)(256 + th_cap + (set.rtab ? std::min(th_cap, kRowTabMax / 4) : 0)) * 4;
}

cudaError_t launch_prep(const Set& set, const Items& it, const Plan& pl, float* tables, uint64_t* sums,
                        bool early, int sm_count, LaunchCache& lc, cudaStream_t s, int th_cap) {
  if (it.n <= 0) return cudaSuccess;
  const Dims& d = set.d;
  const int cap = th_cap > 0 && th_cap < d.theta_cap && set.rtab && d.K4 * th_cap <= kRowTabMax ? th_cap
                                                                                                   : d.theta_cap;
  const size_t smem = prep_smem_bytes(set, cap);
  const int fl = lc.floors ? 1 : 0, mode = fl + (set.prior == 1 ? 2 : 0);
  auto kern = mode == 0 ? k_prep<false, false> : mode == 1 ? k_prep<true, false>
            : mode == 2 ? k_prep<false, true> : k_prep<true, true>;
  if (smem > lc.prep_smem[mode]) {
    cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), smem);
    if (e != cudaSuccess) return e;
    lc.prep_smem[mode] = smem;
  }
  // (five 256-thread blocks fit an SM by registers; 64-thread blocks need at
  // least 64 threads for the classes' demands, K <= 64)
  const int tb = (long long)it.n * 2 > 2LL * 5 * sm_count ? 64 : kPrepThreads;
  return launch_pdl(kern, dim3(it.n * 2), dim3(tb), smem, s, set, it, pl, tables, sums, early ? 1 : 0, cap);
}

static int score_lcap(const Dims& d) { return d.lcap < kSmemTableCap ? d.lcap : kSmemTableCap; }

cudaError_t launch_score(const Set& set, const Items& it, const Plan& pl, const float* tables, uint64_t* sums,
                         void* dump, int dump_stride, int sm_count, LaunchCache& lc, cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  ScoreGrid sg{};
  sg.lcap_s = score_lcap(set.d);
  sg.tcopy = kTableHeader + 3 * sg.lcap_s;
  // the table path when a segment's W + 1 entries cost well under a chunk's
  // samples (an entry costs about one scenario of the plain path, a scenario
  // about a third of one there); the smallest chunk holds 2 calls per thread
  const long long chunk_min = std::min<long long>(pl.S, 2LL * 4 * kScoreThreads);
  const bool table = !dump && pl.W <= 4096 && 3LL * (pl.W + 1) <= 2 * chunk_min;
  const bool rf = set.prior == 1;
  const size_t stages = 16 + 2 * (size_t)(pl.Wp + 2 * sg.tcopy) * 4;
  const size_t gt_len = rf ? 2 * (size_t)pl.W : (size_t)pl.W + 1;
  const size_t smem = stages + (table ? ((it.p == nullptr ? 2 : 1) * 8 * gt_len + 15) / 16 * 16 : 0);
  const int v = dump ? SCORE_DUMP : table ? (it.p == nullptr ? SCORE_TABLE : SCORE_TABLE_MULTI) : SCORE_PLAIN;
  const int fl = lc.floors ? 1 : 0, mode = fl + (rf ? 2 : 0);
  const bool one = it.p == nullptr;  // every item belongs to problem 0
#define FS_KERN(F, R)                                                                              \
  (dump ? k_score<true, F, false, false, R>                                                         \
        : table ? (one ? k_score<false, F, true, true, R> : k_score<false, F, true, false, R>)      \
                : k_score<false, F, false, false, R>)
  auto kern = mode == 0 ? FS_KERN(false, false) : mode == 1 ? FS_KERN(true, false)
            : mode == 2 ? FS_KERN(false, true) : FS_KERN(true, true);
#undef FS_KERN
  const void* kfun = reinterpret_cast<const void*>(kern);
  if (smem != lc.score_smem[v][mode]) {
    cudaError_t e = raise_smem_limit(kfun, smem);
    for (int b = 0; b < 3 && e == cudaSuccess; ++b) {
      int per_sm = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kfun, kScoreThreads >> b, smem);
      lc.score_blocks_per_sm[v][mode][b] = per_sm < 1 ? 1 : per_sm;
    }
    if (e != cudaSuccess) return e;
    lc.score_smem[v][mode] = smem;
  }
  // Chunks of U calls per thread: about eight chunks per resident block when
  // the work allows, so that the counter can even out the segments' unequal
  // costs; at least 2 (a chunk's set-up is then paid for eight samples per
  // thread, measured faster on small launches) and at most 8 calls per
  // thread, and no more than a segment holds.
  int bt = kScoreThreads;
  long long resident = (long long)lc.score_blocks_per_sm[v][mode][0] * sm_count;
  const long long total_calls = (long long)it.n * pl.O * pl.calls;
  long long U = total_calls / ((long long)bt * resident * 8);
  long long u_seg = ((long long)pl.calls + bt - 1) / bt;
  if (U > 8) U = 8;
  if (U < 2) U = 2;
  if (U > u_seg) U = u_seg;
  if (table) {
    // Every chunk pays a fixed set-up (its records' wait, header reads, the
    // barrier, the reduction and its atomic) and builds its segment's table
    // before it draws. Pick the block size (256 or 128 threads; also 64 over
    // several problems, whose segments are short: on one problem's long
    // segments 64-thread blocks, each holding a full block's shared memory,
    // measured slower than the model says) and the chunk
    // length (up to 4096 calls per chunk) that minimise rounds of chunks per
    // block x resident threads per SM x (set-up + build + draws), in units of
    // about one thread-instruction: set-up ~180 per thread, an entry ~60 per
    // thread share, a call's four draws ~72. Smaller blocks give each thread
    // more of a segment's calls, so the set-up is paid fewer times.
    const long long n_seg = (long long)it.n * pl.O;
    long long best = -1;
    for (int b = 0; b < (one ? 2 : 3); ++b) {
      const int tb = kScoreThreads >> b;
      const long long res_b = (long long)lc.score_blocks_per_sm[v][mode][b] * sm_count;
      const long long us_b = ((long long)pl.calls + tb - 1) / tb;
      const long long build = ((pl.W + 1 + tb - 1) / tb) * 60;
      const long long u_hi = std::min<long long>(4096 / tb, us_b);
      for (long long u = std::min<long long>(2, us_b); u <= u_hi; ++u) {
        const long long nch_u = (pl.calls + tb * u - 1) / (tb * u);
        const long long rounds = (n_seg * nch_u + res_b - 1) / res_b;
        const long long cost = rounds * lc.score_blocks_per_sm[v][mode][b] * tb * (180 + build + 72 * u);
        if (best < 0 || cost < best) {
          best = cost;
          U = u;
          bt = tb;
          resident = res_b;
          u_seg = us_b;
        }
      }
    }
  }
  // chunk indices are 32-bit: widen the chunks until they fit (one chunk per
  // segment gives n O <= 2^30 chunks, which the entry points guarantee)
  long long nch = (pl.calls + bt * U - 1) / (bt * U);
  while ((long long)it.n * pl.O * nch >= (1LL << 31) && U < u_seg) {
    U *= 2;
    nch = (pl.calls + bt * U - 1) / (bt * U);
  }
  if ((long long)it.n * pl.O * nch >= (1LL << 31)) return cudaErrorInvalidValue;
  sg.chunk = (int)(bt * U);
  sg.nch = (int)nch;
  sg.total = (int)((long long)it.n * pl.O * nch);
  const int grid = (int)(sg.total < resident ? sg.total : resident);
  sg.dyn = sg.total >= 4LL * grid ? 1 : 0;
  return launch_pdl(kern, dim3(grid), dim3(bt), smem, s, set, it, pl, tables, sums,
                    (unsigned char*)dump, dump ? dump_stride : 0, sg);
}

int finalize_blocks(const Items& it) {
  if (it.off) return 0;
  const int nb = (it.n + 255) / 256;  // one candidate per thread
  return nb < 2 ? 0 : (nb > kFinalizeMaxBlocks ? kFinalizeMaxBlocks : nb);
}

cudaError_t launch_finalize(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums, double* gap,
                            double* score, float* gamma_t, int32_t* best, uint32_t* status_copy, uint64_t* part,
                            cudaStream_t s) {
  const int nb = finalize_blocks(it);
  if (nb > 0 && part)
    return launch_pdl(k_finalize_split, dim3(nb), dim3(256), 0, s, set, it, pl, sums, gap, score, gamma_t, best,
                      status_copy, part);
  return launch_pdl(k_finalize, dim3(it.off ? set.P : 1), dim3(256), 0, s, set, it, pl, sums, gap, score, gamma_t,
                    best, status_copy);
}

// ---------------------------------------------------------------- measurement floors (not part of the method)

// What the table path's draws cost without the rest of the scorer. MODE 0:
// Philox4x32-10 of the table path's counters alone (two chains a thread, the
// words XORed so that none is dead). MODE 1: the same draws with the table
// path's per-sample work, sample_gtab over a block-local table of W + 1
// entries with the gate the same at every position (position, entry address,
// load and 64-bit sum). No chunks, staging, table builds or barriers: each
// block takes one segment of per_thread calls a thread. One word per thread out.
template <int MODE>
__global__ void __launch_bounds__(kScoreThreads) k_draw_floor(Plan pl, int per_thread, uint64_t* out) {
  extern __shared__ __align__(16) unsigned char smraw[];
  uint64_t* tab = reinterpret_cast<uint64_t*>(smraw);
  for (int k = (int)threadIdx.x; k <= pl.W; k += (int)blockDim.x) tab[k] = (uint64_t)k * 977u;
  __syncthreads();
  const int step = (int)blockDim.x, q_hi = per_thread * step;
  const uint32_t cell = blockIdx.x;
  uint64_t v = 0;
  if constexpr (MODE == 1) {
    const PhiloxKeys keys{};  // not read: one-problem draws take the plan's round keys
    v = sample_gtab<true, false, false>(pl, keys, 0, (int)cell, 0, q_hi, smem_u32(tab), 0u, 8u);
  } else {
    uint32_t acc = 0;
    int q = (int)threadIdx.x;
    for (; q + step < q_hi; q += 2 * step) {
      const uint4 x0 = philox4x32_10_plan(make_uint4((uint32_t)q, 0u, cell, pl.round), pl);
      const uint4 x1 = philox4x32_10_plan(make_uint4((uint32_t)(q + step), 0u, cell, pl.round), pl);
      acc ^= x0.x ^ x0.y ^ x0.z ^ x0.w ^ x1.x ^ x1.y ^ x1.z ^ x1.w;
    }
    if (q < q_hi) {
      const uint4 x = philox4x32_10_plan(make_uint4((uint32_t)q, 0u, cell, pl.round), pl);
      acc ^= x.x ^ x.y ^ x.z ^ x.w;
    }
    v = acc;
  }
  out[(size_t)blockIdx.x * blockDim.x + threadIdx.x] = v;
}

cudaError_t draw_floor(int mode, int w, long long calls, int reps, int sm_count, double* ms_median,
                       long long* calls_done) {
  const int bt = kScoreThreads / 2;  // the table path's blocks on large launches
  auto kern = mode == 0 ? k_draw_floor<0> : k_draw_floor<1>;
  const size_t smem = 8 * (((size_t)1 << w) + 1);
  int per_sm = 0;
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), smem);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, bt, smem);
  if (e != cudaSuccess) return e;
  const long long grid = (long long)(per_sm < 1 ? 1 : per_sm) * sm_count;
  const long long per_thread = (calls + grid * bt - 1) / (grid * bt);
  if (per_thread < 1 || 4 * per_thread * bt > 0x7FFFFFFFLL) return cudaErrorInvalidValue;
  Plan pl{};
  pl.key0 = 0x0F1E2D3Cu;
  pl.key1 = 0x4B5A6978u;
  pl.W = 1 << w;
  pl.w = w;
  pl.S = (int)(4 * per_thread * bt);  // every call of a segment serves four samples
  plan_round_keys(pl);
  uint64_t* out = nullptr;
  cudaEvent_t a = nullptr, b = nullptr;
  std::vector<float> t;
  e = cudaMalloc(&out, (size_t)grid * bt * sizeof(uint64_t));
  if (e == cudaSuccess) e = cudaEventCreate(&a);
  if (e == cudaSuccess) e = cudaEventCreate(&b);
  for (int i = 0; e == cudaSuccess && i < reps + 3; ++i) {  // three untimed launches first
    e = cudaEventRecord(a, 0);
    note_launch();
    if (e == cudaSuccess) kern<<<(unsigned)grid, bt, smem, 0>>>(pl, (int)per_thread, out);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaEventRecord(b, 0);
    if (e == cudaSuccess) e = cudaEventSynchronize(b);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, a, b);
    if (e == cudaSuccess && i >= 3) t.push_back(ms);
  }
  if (a) cudaEventDestroy(a);
  if (b) cudaEventDestroy(b);
  if (out) cudaFree(out);
  if (e != cudaSuccess) return e;
  std::sort(t.begin(), t.end());
  *ms_median = t[t.size() / 2];
  *calls_done = grid * bt * per_thread;
  return cudaSuccess;
}

}  // namespace fs
