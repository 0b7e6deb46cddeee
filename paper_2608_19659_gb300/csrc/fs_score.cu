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
//
// k_prep builds, per (candidate, realisation), the part of that table a
// scenario can reach: Theta entries with kappa in (Cexcl, max(Cexcl, cap_hi_e)].
// k_score draws each scenario (Philox4x32-10 + quantile lookup), evaluates
// both t* by a binary search of the staged table plus one fulfilment, and
// sums g = rint(Gamma' 2^40) in int64. k_finalize turns the sums into
// E[Gamma_{t+1} | e], the score and the argmax.
#include <cuda_runtime.h>

#include "fs_finalize.cuh"
#include "fs_internal.cuh"

namespace fs {

// Budget left for class ie and its cheapest cover without row rr, at threshold t.
struct Eval {
  int A;   // -1 if another class has no cover
  int P;   // kCostInf if no other row of class ie covers t
};

__device__ __forceinline__ Eval warp_eval_excl(float t, const float* sC, const float* sLam, const float* sRl,
                                               const Dims& d, int rr, int ie, int lane) {
  int R = 0;
  bool rinf = false;
  int P = kCostInf;
  for (int base = 0; base < d.K4; base += 32) {
    const int rho = base + lane;
    int cost = kCostInf;
    if (rho < d.K4 && rho != rr) {
      const int n = min_replicas(t, sC[rho], sLam[rho >> 2], sRl[rho >> 2], d.Mf[rho & 3]);
      if (n) cost = n << (rho & 3);
    }
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 1));
    cost = min(cost, __shfl_xor_sync(0xffffffffu, cost, 2));
    const int cls = rho >> 2;
    const bool head = rho < d.K4 && (lane & 3) == 0 && cls != ie;
    if (__ballot_sync(0xffffffffu, head && cost >= kCostInf)) rinf = true;
    R += __reduce_add_sync(0xffffffffu, (head && cost < kCostInf) ? cost : 0);
    const int ibase = ie * 4;
    if (ibase >= base && ibase < base + 32) P = __shfl_sync(0xffffffffu, cost, ibase - base);
  }
  Eval e;
  e.A = rinf ? -1 : d.G - R;
  e.P = P;
  return e;
}

__device__ __forceinline__ int replicas_left(const Eval& e, int jr, const Dims& d) {
  return (e.A >= (1 << jr)) ? min(e.A >> jr, d.M[jr]) : 0;
}

__device__ __forceinline__ bool feasible_at(const Eval& e, int m, float C, float t, float lam, float rl) {
  return (e.P < kCostInf && e.P <= e.A) || (m >= 1 && fulfil_r((float)m, C, lam, rl) >= t);
}

__global__ void __launch_bounds__(kPrepThreads) k_prep(Set set, Items it, Plan pl, float* tables,
                                                       uint64_t* sums) {
  extern __shared__ __align__(16) unsigned char smraw[];
  float* sC = reinterpret_cast<float*>(smraw);  // [256]
  float* sTh = sC + 256;                          // [theta_cap]
  __shared__ float s_cx, s_cmax;
  __shared__ int s_bx;
  const Dims& d = set.d;  // kernel-parameter space: d.M[j] reads need no local copy
  const int item = blockIdx.x >> 1, sigma = blockIdx.x & 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  pdl_wait();     // thresholds, rows and the zeroed lmax come from k_solve
  pdl_trigger();  // k_score may start launching; it waits for this grid to finish
  const int p = it.p ? it.p[item] : 0;
  const int cell = it.cell[item];
  float* tab = tables + ((size_t)item * 2 + sigma) * d.slot_floats;
  if (sigma == 0)
    for (int o = tid; o < pl.O; o += blockDim.x) sums[(size_t)item * pl.O + o] = 0ull;
  if (cell < 0 || cell >= d.cells) {  // device-side candidate ids are checked here
    if (tid == 0) {
      atomicOr(set.status, ST_CELL);
      for (int k = 0; k < kTableHeader; ++k) tab[k] = 0.0f;
      tab[H_BX] = __int_as_float(-1);
    }
    return;
  }
  const int rr = cell / d.B, be = cell - rr * d.B, ie = rr >> 2, jr = rr & 3;
  const float lam = set.lam[ie], L = set.slo[ie], rl = __frcp_rn(lam);
  __shared__ float sLam[FS_MAX_CLASSES], sRl[FS_MAX_CLASSES];  // demand and RN(1/demand)
  if (tid < d.K) {
    sLam[tid] = set.lam[tid];
    sRl[tid] = __frcp_rn(set.lam[tid]);
  }
  const size_t ps = (size_t)p * 2 + sigma;
  const int total = set.ntheta[ps];
  const float* th_g = set.theta + ps * d.theta_cap;
  for (int rho = tid; rho < d.K4; rho += blockDim.x) sC[rho] = set.rowC[ps * d.K4 + rho];
  for (int k = tid; k < total; k += blockDim.x) sTh[k] = th_g[k];
  const float* bp = set.bounds + (size_t)p * 4 * d.cells;
  const float* capS = bp + (size_t)(sigma ? CAP_HI : CAP_LO) * d.cells;
  const float* tailS = bp + (size_t)(sigma ? TAIL_LO : TAIL_HI) * d.cells;

  // best SLO-feasible capacity of row r without bin b_e (ties: lower bin)
  if (warp == 0) {
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
      s_cmax = fmaxf(s_cx, bp[(size_t)CAP_HI * d.cells + cell]);
    }
  }
  __syncthreads();
  const float cx = s_cx, cmax = s_cmax;
  const int msent = d.K == 1 ? d.M[jr] : 0;  // above every threshold only a lone class can go on

  // b0: last index feasible at Cexcl; b1: last index feasible at max(Cexcl, cap_hi).
  // Joint search: each round every warp probes one index; a probe answers for
  // both capacities, and the warps split whichever intervals are still open.
  __shared__ int s_iv[4], s_probe[8];
  if (tid == 0) {
    s_iv[0] = -1;
    s_iv[1] = total;
    s_iv[2] = -1;
    s_iv[3] = total;
  }
  __syncthreads();
  for (;;) {
    const int lo0 = s_iv[0], hi0 = s_iv[1], lo1 = s_iv[2], hi1 = s_iv[3];
    const bool open0 = hi0 - lo0 > 1, open1 = hi1 - lo1 > 1;
    if (!open0 && !open1) break;
    int lo, hi, part, parts;
    if (open0 && open1) {
      const bool first = warp < nwarp / 2;
      lo = first ? lo0 : lo1;
      hi = first ? hi0 : hi1;
      parts = nwarp / 2 + 1;
      part = (first ? warp : warp - nwarp / 2) + 1;
    } else {
      lo = open0 ? lo0 : lo1;
      hi = open0 ? hi0 : hi1;
      parts = nwarp + 1;
      part = warp + 1;
    }
    int k = lo + (int)(((long long)part * (hi - lo)) / parts);
    k = max(lo + 1, min(hi - 1, k));
    const Eval e = warp_eval_excl(sTh[k], sC, sLam, sRl, d, rr, ie, lane);
    const int m = replicas_left(e, jr, d);
    if (lane == 0) {
      s_probe[2 * warp] = k;
      s_probe[2 * warp + 1] = (feasible_at(e, m, cx, sTh[k], lam, rl) ? 1 : 0) | (feasible_at(e, m, cmax, sTh[k], lam, rl) ? 2 : 0);
    }
    __syncthreads();
    if (tid == 0) {
      int a0 = lo0, c0 = hi0, a1 = lo1, c1 = hi1;
      for (int w = 0; w < nwarp; ++w) {
        const int kk = s_probe[2 * w], f = s_probe[2 * w + 1];
        if (f & 1) a0 = max(a0, kk); else c0 = min(c0, kk);
        if (f & 2) a1 = max(a1, kk); else c1 = min(c1, kk);
      }
      s_iv[0] = a0;
      s_iv[1] = c0;
      s_iv[2] = a1;
      s_iv[3] = c1;
    }
    __syncthreads();
  }
  const int b0 = s_iv[0], b1 = s_iv[2];
  const int Lt = b1 - b0;
  // arrays padded to P = pow2 >= Lt + 1 entries (+inf beyond Lt), so the
  // scenario search needs no bound checks; at least 4 for 16-byte copies
  int P = 1;
  while (P < Lt + 1) P <<= 1;
  const int Lpad = Lt ? max(P, 4) : 0;
  if (Lpad > d.lcap) {  // cannot happen: Lt <= total <= theta_cap
    if (tid == 0) atomicOr(set.status, ST_TABLE);
    return;
  }
  float* kap = tab + kTableHeader;
  float* tht = kap + Lpad;
  float* mn = tht + Lpad;

  // u = 0..Lt: m at index b0+1+u (m_first, then m_next[u-1]); kappa for u < Lt
  for (int u = warp; u <= Lt; u += nwarp) {
    const int k = b0 + 1 + u;
    int m;
    if (k < total) {
      const Eval e = warp_eval_excl(sTh[k], sC, sLam, sRl, d, rr, ie, lane);
      m = replicas_left(e, jr, d);
    } else {
      m = msent;
    }
    if (u < Lt) {
      // smallest capacity in (cx, cmax] at which f(m, C) >= theta_k, on the bit
      // patterns of nonnegative floats (ordered like the values). First the 32
      // patterns around the real solution t lambda / m, one per lane; if the
      // answer is not among them, a 32-ary search over the whole interval.
      const float t = sTh[k];
      const uint32_t bx = __float_as_uint(cx), bmax = __float_as_uint(cmax);
      const float c0 = __fdiv_rn(__fmul_rn(t, lam), (float)m);
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
        tht[u] = t;
      }
    }
    if (lane == 0) {
      if (u == 0) tab[H_M_FIRST] = (float)m; else mn[u - 1] = (float)m;
    }
  }
  for (int u = Lt + tid; u < Lpad; u += blockDim.x) {
    kap[u] = __int_as_float(0x7f800000);
    tht[u] = 0.0f;
    mn[u] = 0.0f;
  }
  if (tid == 0) {
    tab[H_TH_BASE] = b0 >= 0 ? sTh[b0] : 0.0f;
    tab[H_L] = __int_as_float(Lt);
    tab[H_LPAD] = __int_as_float(Lpad);
    tab[H_CX] = cx;
    tab[H_BX] = __int_as_float(s_bx);
    tab[H_CMAX] = cmax;
    tab[H_LAM] = lam;
    tab[H_LO_C] = bp[(size_t)CAP_LO * d.cells + cell];
    tab[H_HI_C] = bp[(size_t)CAP_HI * d.cells + cell];
    tab[H_LO_L] = bp[(size_t)TAIL_LO * d.cells + cell];
    tab[H_HI_L] = bp[(size_t)TAIL_HI * d.cells + cell];
    tab[H_SLO] = L;
    tab[H_CELL] = __int_as_float(cell);
    tab[H_P] = __int_as_float(p);
    tab[H_STEP0] = __int_as_float(Lt ? P >> 1 : 0);
    atomicMax(set.lmax, Lpad);
  }
}

// t* of one realisation with row capacity C (see the file comment). kap is
// padded with +inf to a power of two above the entry count, so the
// branch-free search needs no bound checks; step0 = half that power.
__device__ __forceinline__ float tstar_of(float C, const float* kap, const float* tht, const float* mn,
                                          int step0, float th_base, float m_first, float lam,
                                          float rlam) {
  int pos = 0;
  for (int step = step0; step > 0; step >>= 1) pos += kap[pos + step - 1] <= C ? step : 0;
  const float thb = pos ? tht[pos - 1] : th_base;
  const float m = pos ? mn[pos - 1] : m_first;
  // the row term is rarely needed; the out-of-line IEEE divide keeps it behind
  // the branch (an inline quotient would be computed for every scenario)
  (void)rlam;
  const float tr = m >= 1.0f ? fulfil(m, C, lam) : 0.0f;
  return tr > thb ? tr : thb;
}

// Per-class choice of one scenario at threshold t (dump mode only): rows from
// the base realisation except row rr, which has capacity C and bin bC.
__device__ void dump_choices(float t, const Set& set, size_t ps, int rr, float C, int bC,
                             uint32_t* choice, int32_t* total_gpus) {
  const Dims& d = set.d;
  int total = 0;
  for (int i = 0; i < d.K; ++i) {
    uint32_t code = 0;
    if (t > 0.0f) {
      int best = kCostInf, bj = -1, bn = 0, bbin = -1;
      for (int j = 0; j < kT; ++j) {
        const int rho = 4 * i + j;
        const float c = rho == rr ? C : set.rowC[ps * d.K4 + rho];
        const int b = rho == rr ? bC : set.rowB[ps * d.K4 + rho];
        if (b < 0) continue;
        const int n = min_replicas(t, c, set.lam[i], __frcp_rn(set.lam[i]), d.Mf[j]);
        if (n && (n << j) < best) {
          best = n << j;
          bj = j;
          bn = n;
          bbin = b;
        }
      }
      if (bj >= 0) {
        code = (uint32_t)bn | ((uint32_t)bj << 16) | ((uint32_t)bbin << 18);
        total += best;
      }
    }
    choice[i] = code;
  }
  *total_gpus = t > 0.0f ? total : 0;
}

// Philox calls [q_lo, q_hi) of one (candidate, outcome) segment; call q
// serves samples 4q..4q+3, sample 4q+h reading output word h (upper 16 bits:
// capacity position, lower 16 bits: tail position; top log2(W) bits each).
// h0/h1 point at the staged table headers; kap/tht/mnn at the table arrays
// (shared memory when TS, else global). Without DUMP, sQ holds the stratum's
// capacities already mapped into [cap_lo, cap_hi], and the tail gate of
// Eq. 5 (l_y <= L_i) is the position test kl < kgate (the mapped tail
// quantiles are nondecreasing in the position); with DUMP, sQ holds the raw
// quantiles and both values are mapped per sample.
template <bool DUMP, bool TS>
__device__ __forceinline__ uint64_t run_piece(const Set& set, const Plan& pl, int item, int o, int q_lo,
                                              int q_hi, const float* sQ, int qoff, int kgate, const float* h0,
                                              const float* h1, const float* kap0, const float* tht0,
                                              const float* mn0, const float* kap1, const float* tht1,
                                              const float* mn1, unsigned char* dump, int dump_stride) {
  const int st0 = __float_as_int(h0[H_STEP0]), st1 = __float_as_int(h1[H_STEP0]);
  const float thb0 = h0[H_TH_BASE], mf0 = h0[H_M_FIRST], cx0 = h0[H_CX];
  const float thb1 = h1[H_TH_BASE], mf1 = h1[H_M_FIRST], cx1 = h1[H_CX];
  const float lam = h0[H_LAM], rlam = __frcp_rn(lam);
  const int cell = __float_as_int(h0[H_CELL]), p = __float_as_int(h0[H_P]);
  const PhiloxKeys keys = philox_keys(pl.key0, pl.key1 ^ (pl.stream_base + (uint32_t)p));
  const uint32_t sh = (uint32_t)pl.sh;
  const int S = pl.S;
  const uint32_t ctr1 = (uint32_t)o, ctr2 = (uint32_t)cell, ctr3 = pl.round;
  const float* sQo = sQ + qoff;
  uint64_t acc = 0;
  for (int q = q_lo + (int)threadIdx.x; q < q_hi; q += blockDim.x) {
    const uint4 x = philox4x32_10(make_uint4((uint32_t)q, ctr1, ctr2, ctr3), keys);
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const int s = 4 * q + h;
      const uint32_t word = h == 0 ? x.x : h == 1 ? x.y : h == 2 ? x.z : x.w;
      const int kc = (int)((word >> 16) >> sh);
      const int kl = (int)((word & 0xFFFFu) >> sh);
      float cy, ly = 0.0f;
      bool gate;
      if (DUMP) {
        const float lo_c = h0[H_LO_C], hi_c = h0[H_HI_C], lo_l = h0[H_LO_L], hi_l = h0[H_HI_L];
        cy = map_into(lo_c, __fsub_rn(hi_c, lo_c), hi_c, sQo[kc]);
        ly = map_into(lo_l, __fsub_rn(hi_l, lo_l), hi_l, sQo[kl]);
        gate = ly <= h0[H_SLO];
      } else {
        cy = sQo[kc];
        gate = kl < kgate;
      }
      const float C0 = gate ? fmaxf(cx0, cy) : cx0;
      const float C1 = gate ? fmaxf(cx1, cy) : cx1;
      const float t0 = tstar_of(C0, kap0, tht0, mn0, st0, thb0, mf0, lam, rlam);
      const float t1 = tstar_of(C1, kap1, tht1, mn1, st1, thb1, mf1, lam, rlam);
      const uint64_t gf = fixed40(__fsub_rn(t1, t0));
      acc += (h == 0 || s < S) ? gf : 0ull;  // the last call may serve fewer than four samples
      if (DUMP && (h == 0 || s < S)) {
        const size_t idx = ((size_t)item * pl.O + o) * pl.S + s;
        unsigned char* rec = dump + idx * dump_stride;
        fs_scenario_head hd;
        hd.c_y = cy;
        hd.l_y = ly;
        hd.t_star[0] = t0;
        hd.t_star[1] = t1;
        const int rr = cell / set.d.B, be = cell - rr * set.d.B;
        uint32_t* ch = reinterpret_cast<uint32_t*>(rec + sizeof(fs_scenario_head));
#pragma unroll
        for (int sg = 0; sg < 2; ++sg) {
          const float cx = sg ? cx1 : cx0;
          const int bx = __float_as_int(sg ? h1[H_BX] : h0[H_BX]);
          int bC;
          if (!gate) bC = bx;
          else if (bx < 0 || cy > cx) bC = be;
          else if (cy == cx) bC = min(be, bx);
          else bC = bx;
          dump_choices(sg ? t1 : t0, set, (size_t)p * 2 + sg, rr, sg ? C1 : C0, bC, ch + sg * set.d.K,
                       &hd.total_gpus[sg]);
        }
        *reinterpret_cast<fs_scenario_head*>(rec) = hd;
      }
    }
  }
  return acc;
}

// Thread 0: stage segment seg (its quantile window and both candidate tables,
// header plus lcopy entries each) into dst, completing on bar.
__device__ __forceinline__ void stage_segment(const Set& set, const Plan& pl, const float* tables, int seg,
                                              float* dst, uint64_t* bar, int qwin, int tstride, int lcopy) {
  const Dims& d = set.d;
  const int item = seg / pl.O, o = seg - item * pl.O;
  const int q0 = (o * pl.W) & ~3;
  const int q1 = min(((o + 1) * pl.W + 3) & ~3, d.Q);
  const float* tab = tables + (size_t)item * 2 * d.slot_floats;
  const uint32_t tb = (uint32_t)(kTableHeader + 3 * lcopy) * 4u;
  const uint32_t qb = (uint32_t)(q1 - q0) * 4u;
  fence_proxy_async();
  mbar_expect_tx(bar, qb + 2 * tb);
  bulk_g2s(dst, set.qn + q0, qb, bar);
  bulk_g2s(dst + qwin, tab, tb, bar);
  bulk_g2s(dst + qwin + tstride, tab + d.slot_floats, tb, bar);
}

// Each block owns a contiguous range of the flattened Philox-call index
// (segment = (candidate, outcome), ceil(S/4) calls each), so the work is
// balanced to within one call per thread. A segment's quantile window and
// both candidate tables are staged in shared memory by TMA bulk copies,
// double-buffered: the next segment's copies fly while this one computes.
template <bool DUMP>
__global__ void __launch_bounds__(kScoreThreads, 5) k_score(Set set, Items it, Plan pl, const float* tables,
                                                         uint64_t* sums, unsigned char* dump, int dump_stride,
                                                         long long total_calls, int lcap_s, int qwin) {
  extern __shared__ __align__(16) unsigned char smraw[];
  uint64_t* bar = reinterpret_cast<uint64_t*>(smraw);  // [2]
  const int tstride = kTableHeader + 3 * lcap_s;
  const int stage_floats = qwin + 2 * tstride;
  float* stage0 = reinterpret_cast<float*>(smraw + 16);
  __shared__ int s_lcopy;
  const Dims& d = set.d;  // kernel-parameter space: d.M[j] reads need no local copy
  const int tid = threadIdx.x, lane = tid & 31;

  pdl_wait();  // tables, zeroed sums and lmax come from k_prep
  const long long g = gridDim.x;
  const long long r_lo = total_calls * blockIdx.x / g;
  const long long r_hi = total_calls * (blockIdx.x + 1) / g;
  if (r_hi <= r_lo) return;
  const int seg_first = (int)(r_lo / pl.calls);
  const int seg_last = (int)((r_hi - 1) / pl.calls);

  if (tid == 0) {
    s_lcopy = min(*set.lmax, lcap_s);
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
  }
  __syncthreads();
  const int lcopy = s_lcopy;
  if (tid == 0) stage_segment(set, pl, tables, seg_first, stage0, bar, qwin, tstride, lcopy);

  int j = 0;
  for (int seg = seg_first; seg <= seg_last; ++seg, ++j) {
    const int st = j & 1;
    if (tid == 0 && seg < seg_last)
      stage_segment(set, pl, tables, seg + 1, stage0 + (size_t)(st ^ 1) * stage_floats, bar + (st ^ 1), qwin,
                    tstride, lcopy);
    const bool ok = mbar_wait(&bar[st], (uint32_t)((j >> 1) & 1), kWaitLimitNs);
    if (__syncthreads_or(!ok)) {
      if (tid == 0) atomicOr(set.status, ST_TIMEOUT);
      // let copies in flight land before the block exits (bounded as well)
      mbar_wait(&bar[st], (uint32_t)((j >> 1) & 1), kWaitLimitNs);
      if (seg < seg_last) mbar_wait(&bar[st ^ 1], (uint32_t)(((j + 1) >> 1) & 1), kWaitLimitNs);
      return;
    }
    float* stg = stage0 + (size_t)st * stage_floats;
    const float* h0 = stg + qwin;
    const float* h1 = h0 + tstride;
    const int item = seg / pl.O, o = seg - item * pl.O;
    const long long sb = (long long)seg * pl.calls;
    const int q_lo = (int)(max(r_lo, sb) - sb);
    const int q_hi = (int)(min(r_hi, sb + pl.calls) - sb);
    const int qoff = o * pl.W - ((o * pl.W) & ~3);
    const int Lp0 = __float_as_int(h0[H_LPAD]), Lp1 = __float_as_int(h1[H_LPAD]);
    const int cell = __float_as_int(h0[H_CELL]);
    const bool cell_ok = cell >= 0 && cell < d.cells;  // a bad device-side id was flagged by k_prep
    int kgate = 0;
    if (!DUMP) {
      // map the stratum's quantiles into this cell's capacity interval in place,
      // and count the positions whose tail value passes the SLO gate
      const float lo_c = h0[H_LO_C], hi_c = h0[H_HI_C], lo_l = h0[H_LO_L], hi_l = h0[H_HI_L];
      const float d_c = __fsub_rn(hi_c, lo_c), d_l = __fsub_rn(hi_l, lo_l), slo = h0[H_SLO];
      for (int k0 = 0; k0 < pl.W; k0 += blockDim.x) {
        const int k = k0 + tid;
        bool pass = false;
        if (k < pl.W) {
          const float qv = stg[qoff + k];
          stg[qoff + k] = map_into(lo_c, d_c, hi_c, qv);
          pass = map_into(lo_l, d_l, hi_l, qv) <= slo;
        }
        kgate += __syncthreads_count(pass);
      }
    }
    uint64_t acc = 0;
    if (cell_ok) {
      if (Lp0 <= lcopy && Lp1 <= lcopy) {
        acc = run_piece<DUMP, true>(set, pl, item, o, q_lo, q_hi, stg, qoff, kgate, h0, h1, h0 + kTableHeader,
                                    h0 + kTableHeader + Lp0, h0 + kTableHeader + 2 * Lp0, h1 + kTableHeader,
                                    h1 + kTableHeader + Lp1, h1 + kTableHeader + 2 * Lp1, dump, dump_stride);
      } else {
        const float* g0 = tables + (size_t)item * 2 * d.slot_floats + kTableHeader;
        const float* g1 = g0 + d.slot_floats;
        acc = run_piece<DUMP, false>(set, pl, item, o, q_lo, q_hi, stg, qoff, kgate, h0, h1, g0, g0 + Lp0,
                                     g0 + 2 * Lp0, g1, g1 + Lp1, g1 + 2 * Lp1, dump, dump_stride);
      }
    }
    for (int off = 16; off; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
    if (lane == 0 && acc)
      atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)seg]), (unsigned long long)acc);
    __syncthreads();  // stage st is free for the copies issued next iteration
  }
  pdl_trigger();
}

__global__ void k_finalize(Set set, Items it, Plan pl, const uint64_t* sums, double* gap, double* score,
                           float* gamma_t, int32_t* best) {
  pdl_wait();
  const int p = blockIdx.x;
  const int beg = it.off ? it.off[p] : 0;
  const int end = it.off ? it.off[p + 1] : it.n;
  const Best b = finalize_problem(set, it, pl, sums, p, beg, end, gap, score, gamma_t ? gamma_t + p : nullptr);
  if (threadIdx.x == 0 && best) best[p] = b.pos >= 0 ? it.cell[beg + b.pos] : -1;
}

static size_t prep_smem_bytes(const Dims& d) { return (size_t)(256 + d.theta_cap) * 4; }

cudaError_t launch_prep(const Set& set, const Items& it, const Plan& pl, float* tables, uint64_t* sums,
                        LaunchCache& lc, cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  const size_t smem = prep_smem_bytes(set.d);
  if (smem > lc.prep_smem) {
    cudaError_t e = cudaFuncSetAttribute(k_prep, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    lc.prep_smem = smem;
  }
  return launch_pdl(k_prep, dim3(it.n * 2), dim3(kPrepThreads), smem, s, set, it, pl, tables, sums);
}

static int score_lcap(const Dims& d) { return d.lcap < kSmemTableCap ? d.lcap : kSmemTableCap; }

static int score_qwin(const Dims& d, const Plan& pl) {
  const int w = ((pl.W + 3) & ~3) + 4;
  return w < d.Q ? w : d.Q;
}

cudaError_t launch_score(const Set& set, const Items& it, const Plan& pl, const float* tables, uint64_t* sums,
                         void* dump, int dump_stride, int sm_count, LaunchCache& lc, cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  const long long total = (long long)it.n * pl.O * pl.calls;
  const int lcap_s = score_lcap(set.d), qwin = score_qwin(set.d, pl);
  const size_t smem = 16 + 2 * (size_t)(qwin + 2 * (kTableHeader + 3 * lcap_s)) * 4;
  const int v = dump ? 1 : 0;
  if (smem != lc.score_smem[v]) {
    cudaError_t e;
    int per_sm = 0;
    if (dump) {
      e = cudaFuncSetAttribute(k_score<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_score<true>, kScoreThreads, smem);
    } else {
      e = cudaFuncSetAttribute(k_score<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_score<false>, kScoreThreads, smem);
    }
    if (e != cudaSuccess) return e;
    lc.score_smem[v] = smem;
    lc.score_blocks_per_sm[v] = per_sm < 1 ? 1 : per_sm;
  }
  // One resident wave at least; up to four when every block still gets >= 16
  // calls per thread, so that the block scheduler evens out segments of
  // unequal cost (table length, fulfilment divisions).
  const long long resident = (long long)lc.score_blocks_per_sm[v] * sm_count;
  const long long by_work = total / ((long long)kScoreThreads * 16);
  long long grid_l = by_work < 4 * resident ? by_work : 4 * resident;
  if (grid_l < resident) grid_l = resident;
  const long long min_blocks = (total + kScoreThreads - 1) / kScoreThreads;
  if (grid_l > min_blocks) grid_l = min_blocks;
  const int grid = (int)grid_l;
  if (dump)
    return launch_pdl(k_score<true>, dim3(grid), dim3(kScoreThreads), smem, s, set, it, pl, tables, sums,
                      (unsigned char*)dump, dump_stride, total, lcap_s, qwin);
  return launch_pdl(k_score<false>, dim3(grid), dim3(kScoreThreads), smem, s, set, it, pl, tables, sums,
                    (unsigned char*)nullptr, 0, total, lcap_s, qwin);
}

cudaError_t launch_finalize(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums, double* gap,
                            double* score, float* gamma_t, int32_t* best, cudaStream_t s) {
  return launch_pdl(k_finalize, dim3(it.off ? set.P : 1), dim3(256), 0, s, set, it, pl, sums, gap, score,
                    gamma_t, best);
}

}  // namespace fs
