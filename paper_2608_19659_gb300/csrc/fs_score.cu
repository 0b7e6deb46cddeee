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

#include "fs_internal.cuh"
#include "fs_finalize.cuh"

namespace fs {

// Budget left for class ie and its cheapest cover without row rr, at threshold t.
struct Eval {
  int A;   // -1 if another class has no cover
  int P;   // kCostInf if no other row of class ie covers t
};

__device__ __forceinline__ Eval warp_eval_excl(float t, const float* sC, const float* lam,
                                               const Dims& d, int rr, int ie, int lane) {
  int R = 0;
  bool rinf = false;
  int P = kCostInf;
  for (int base = 0; base < d.K4; base += 32) {
    const int rho = base + lane;
    int cost = kCostInf;
    if (rho < d.K4 && rho != rr) {
      const int n = min_replicas(t, sC[rho], lam[rho >> 2], d.M[rho & 3]);
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

__device__ __forceinline__ bool feasible_at(const Eval& e, int m, float C, float t, float lam) {
  return (e.P < kCostInf && e.P <= e.A) || (m >= 1 && fulfil((float)m, C, lam) >= t);
}

__global__ void __launch_bounds__(kPrepThreads) k_prep(Set set, Items it, Plan pl, float* tables,
                                                       uint64_t* sums) {
  __shared__ float sC[256];
  __shared__ float s_cx, s_cmax;
  __shared__ int s_bx, s_b0, s_b1;
  const Dims d = set.d;
  const int item = blockIdx.x >> 1, sigma = blockIdx.x & 1;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const int p = it.p ? it.p[item] : 0;
  const int cell = it.cell[item];
  if (sigma == 0)
    for (int o = tid; o < pl.O; o += blockDim.x) sums[(size_t)item * pl.O + o] = 0ull;
  if (cell < 0 || cell >= d.cells) {  // device-side candidate ids are checked here
    if (tid == 0) {
      atomicOr(set.status, ST_CELL);
      float* tab = tables + ((size_t)item * 2 + sigma) * d.slot_floats;
      for (int k = 0; k < kTableHeader; ++k) tab[k] = 0.0f;
      tab[5] = __int_as_float(-1);
    }
    return;
  }
  const int rr = cell / d.B, be = cell - rr * d.B, ie = rr >> 2, jr = rr & 3;
  const float lam = set.lam[ie], L = set.slo[ie];
  const size_t ps = (size_t)p * 2 + sigma;
  for (int rho = tid; rho < d.K4; rho += blockDim.x) sC[rho] = set.rowC[ps * d.K4 + rho];
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
  const int total = set.ntheta[ps];
  const float* th = set.theta + ps * d.theta_cap;
  const int msent = d.K == 1 ? d.M[jr] : 0;  // above every threshold only a lone class can go on

  // b0: last index feasible at Cexcl; b1: last index feasible at max(Cexcl, cap_hi)
  if (warp == 0) {
    int lo = -1, hi = total;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      const Eval e = warp_eval_excl(th[mid], sC, set.lam, d, rr, ie, lane);
      if (feasible_at(e, replicas_left(e, jr, d), cx, th[mid], lam)) lo = mid; else hi = mid;
    }
    const int b0 = lo;
    hi = total;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      const Eval e = warp_eval_excl(th[mid], sC, set.lam, d, rr, ie, lane);
      if (feasible_at(e, replicas_left(e, jr, d), cmax, th[mid], lam)) lo = mid; else hi = mid;
    }
    if (lane == 0) {
      s_b0 = b0;
      s_b1 = lo;
    }
  }
  __syncthreads();
  const int b0 = s_b0, b1 = s_b1;
  const int Lt = b1 - b0;
  float* tab = tables + ((size_t)item * 2 + sigma) * d.slot_floats;
  if (Lt > d.lcap) {  // cannot happen: Lt <= total <= theta_cap <= lcap
    if (tid == 0) atomicOr(set.status, ST_TABLE);
    return;
  }
  const int Lpad = (Lt + 3) & ~3;
  float* kap = tab + kTableHeader;
  float* tht = kap + Lpad;
  float* mn = tht + Lpad;

  // u = 0..Lt: m at index b0+1+u (m_first, then m_next[u-1]); kappa for u < Lt
  for (int u = warp; u <= Lt; u += nwarp) {
    const int k = b0 + 1 + u;
    int m;
    if (k < total) {
      const Eval e = warp_eval_excl(th[k], sC, set.lam, d, rr, ie, lane);
      m = replicas_left(e, jr, d);
    } else {
      m = msent;
    }
    if (u < Lt) {
      // smallest capacity in (cx, cmax] at which f(m, C) >= theta_k: 32-ary search on the
      // bit patterns of nonnegative floats (ordered like the values)
      const float t = th[k];
      uint32_t lo = __float_as_uint(cx), hi = __float_as_uint(cmax);
      while (hi - lo > 1) {
        const uint32_t span = hi - lo;
        const uint32_t pt = lo + (uint32_t)(((uint64_t)(lane + 1) * span) >> 5);
        const bool ok = fulfil((float)m, __uint_as_float(pt), lam) >= t;
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
      if (u == 0) tab[1] = (float)m; else mn[u - 1] = (float)m;
    }
  }
  for (int u = Lt + tid; u < Lpad; u += blockDim.x) {
    kap[u] = __int_as_float(0x7f800000);
    tht[u] = 0.0f;
    mn[u] = 0.0f;
  }
  if (tid == 0) {
    tab[0] = b0 >= 0 ? th[b0] : 0.0f;
    tab[2] = __int_as_float(Lt);
    tab[3] = __int_as_float(Lpad);
    tab[4] = cx;
    tab[5] = __int_as_float(s_bx);
    tab[6] = cmax;
    tab[7] = 0.0f;
  }
}

// t* of one realisation with row capacity C (see the file comment).
__device__ __forceinline__ float tstar_of(float C, const float* kap, const float* tht, const float* mn,
                                          int L, int step0, float th_base, float m_first, float lam) {
  int pos = 0;
  for (int step = step0; step > 0; step >>= 1)
    if (pos + step <= L && kap[pos + step - 1] <= C) pos += step;
  const float thb = pos ? tht[pos - 1] : th_base;
  const float m = pos ? mn[pos - 1] : m_first;
  const float tr = m >= 1.0f ? fulfil(m, C, lam) : 0.0f;
  return tr > thb ? tr : thb;
}

__device__ __forceinline__ int top_pow2(int L) {
  return L > 0 ? (1 << (31 - __clz(L))) : 0;
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
        const int n = min_replicas(t, c, set.lam[i], d.M[j]);
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

template <bool DUMP>
__global__ void __launch_bounds__(kScoreThreads) k_score(Set set, Items it, Plan pl, const float* tables,
                                                         uint64_t* sums, unsigned char* dump, int dump_stride,
                                                         int n_tiles, int lcap_s, int qwin) {
  extern __shared__ __align__(16) unsigned char smraw[];
  uint64_t* bar = reinterpret_cast<uint64_t*>(smraw);
  float* sQ = reinterpret_cast<float*>(smraw + 16);
  const int tstride = kTableHeader + 3 * lcap_s;
  float* sT[2] = {sQ + qwin, sQ + qwin + tstride};
  const Dims d = set.d;
  const int tid = threadIdx.x, lane = tid & 31;

  if (tid == 0) mbar_init(bar, 1);
  __syncthreads();
  uint32_t phase = 0;

  for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int chunk = tile % pl.chunks;
    const int eo = tile / pl.chunks;
    const int o = eo % pl.O;
    const int item = eo / pl.O;
    const int p = it.p ? it.p[item] : 0;
    const int cell = it.cell[item];
    if (cell < 0 || cell >= d.cells) continue;  // flagged by k_prep; uniform over the block
    const float* tab[2] = {tables + (size_t)item * 2 * d.slot_floats,
                           tables + ((size_t)item * 2 + 1) * d.slot_floats};
    int Lr[2], Lp[2];
    bool inS[2];
#pragma unroll
    for (int sg = 0; sg < 2; ++sg) {
      Lr[sg] = __float_as_int(tab[sg][2]);
      Lp[sg] = __float_as_int(tab[sg][3]);
      inS[sg] = Lp[sg] <= lcap_s;
    }
    const int q0 = (o * pl.W) & ~3;
    const int q1 = min(((o + 1) * pl.W + 3) & ~3, d.Q);

    __syncthreads();  // every thread is done with the previous tile's staged data
    if (tid == 0) {
      fence_proxy_async();
      uint32_t bytes = (uint32_t)(q1 - q0) * 4u;
      uint32_t tb[2];
#pragma unroll
      for (int sg = 0; sg < 2; ++sg) {
        tb[sg] = inS[sg] ? (uint32_t)(kTableHeader + 3 * Lp[sg]) * 4u : (uint32_t)kTableHeader * 4u;
        bytes += tb[sg];
      }
      mbar_expect_tx(bar, bytes);
      bulk_g2s(sQ, set.qn + q0, (uint32_t)(q1 - q0) * 4u, bar);
      bulk_g2s(sT[0], tab[0], tb[0], bar);
      bulk_g2s(sT[1], tab[1], tb[1], bar);
    }
    const bool ok = mbar_wait(bar, phase, kWaitLimitNs);
    phase ^= 1u;
    if (__syncthreads_or(!ok)) {
      if (tid == 0) atomicOr(set.status, ST_TIMEOUT);
      mbar_wait(bar, phase ^ 1u, kWaitLimitNs);  // let copies in flight land before exiting
      return;
    }

    const float* kap[2];
    const float* tht[2];
    const float* mnn[2];
#pragma unroll
    for (int sg = 0; sg < 2; ++sg) {
      const float* base = inS[sg] ? sT[sg] : tab[sg];
      kap[sg] = base + kTableHeader;
      tht[sg] = kap[sg] + Lp[sg];
      mnn[sg] = tht[sg] + Lp[sg];
    }
    const float thb0 = sT[0][0], mf0 = sT[0][1], cx0 = sT[0][4];
    const float thb1 = sT[1][0], mf1 = sT[1][1], cx1 = sT[1][4];
    const int st0 = top_pow2(Lr[0]), st1 = top_pow2(Lr[1]);

    const int ie = cell / d.B >> 2;
    const float lam = set.lam[ie], Lslo = set.slo[ie];
    const float* bp = set.bounds + (size_t)p * 4 * d.cells;
    const float lo_c = bp[(size_t)CAP_LO * d.cells + cell], hi_c = bp[(size_t)CAP_HI * d.cells + cell];
    const float lo_l = bp[(size_t)TAIL_LO * d.cells + cell], hi_l = bp[(size_t)TAIL_HI * d.cells + cell];
    const float d_c = __fsub_rn(hi_c, lo_c), d_l = __fsub_rn(hi_l, lo_l);
    const uint32_t k0 = pl.key0, k1 = pl.key1 ^ (pl.stream_base + (uint32_t)p);
    const int qoff = o * pl.W - q0;
    const uint32_t W = (uint32_t)pl.W;

    uint64_t acc = 0;
    for (int pp = 0; pp < pl.ppt; ++pp) {
      const int pair = (chunk * pl.ppt + pp) * blockDim.x + tid;
      if (pair >= pl.pairs) break;
      const uint4 x = philox4x32_10(make_uint4((uint32_t)pair, (uint32_t)o, (uint32_t)cell, pl.round), k0, k1);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int s = 2 * pair + h;
        if (h == 1 && s >= pl.S) break;
        const uint32_t xc = h ? x.z : x.x;
        const uint32_t xl = h ? x.w : x.y;
        const int kc = qoff + (int)__umulhi(xc, W);  // top log2(W) bits
        const int kl = qoff + (int)__umulhi(xl, W);
        const float cy = map_into(lo_c, d_c, hi_c, sQ[kc]);
        const float ly = map_into(lo_l, d_l, hi_l, sQ[kl]);
        const bool gate = ly <= Lslo;                       // Eq. 5 for the revealed cell
        const float C0 = gate ? fmaxf(cx0, cy) : cx0;
        const float C1 = gate ? fmaxf(cx1, cy) : cx1;
        const float t0 = tstar_of(C0, kap[0], tht[0], mnn[0], Lr[0], st0, thb0, mf0, lam);
        const float t1 = tstar_of(C1, kap[1], tht[1], mnn[1], Lr[1], st1, thb1, mf1, lam);
        const float g = __fsub_rn(t1, t0);
        acc += (uint64_t)__float2ll_rn(__fmul_rn(g, 0x1p40f));
        if (DUMP) {
          const size_t idx = ((size_t)item * pl.O + o) * pl.S + s;
          unsigned char* rec = dump + idx * dump_stride;
          fs_scenario_head hd;
          hd.c_y = cy;
          hd.l_y = ly;
          hd.t_star[0] = t0;
          hd.t_star[1] = t1;
          const int rr = cell / d.B, be = cell - rr * d.B;
          uint32_t* ch = reinterpret_cast<uint32_t*>(rec + sizeof(fs_scenario_head));
#pragma unroll
          for (int sg = 0; sg < 2; ++sg) {
            const float cx = sg ? cx1 : cx0;
            const int bx = __float_as_int(sg ? sT[1][5] : sT[0][5]);
            const float C = sg ? C1 : C0;
            int bC;
            if (!gate) bC = bx;
            else if (bx < 0 || cy > cx) bC = be;
            else if (cy == cx) bC = min(be, bx);
            else bC = bx;
            dump_choices(sg ? t1 : t0, set, (size_t)p * 2 + sg, rr, C, bC, ch + sg * d.K,
                         &hd.total_gpus[sg]);
          }
          *reinterpret_cast<fs_scenario_head*>(rec) = hd;
        }
      }
    }
    for (int off = 16; off; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
    if (lane == 0 && acc)
      atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)item * pl.O + o]),
                (unsigned long long)acc);
  }
}

__global__ void k_finalize(Set set, Items it, Plan pl, const uint64_t* sums, double* gap, double* score,
                           float* gamma_t, int32_t* best) {
  const int p = blockIdx.x;
  const int beg = it.off ? it.off[p] : 0;
  const int end = it.off ? it.off[p + 1] : it.n;
  const Best b = finalize_problem(set, it, pl, sums, p, beg, end, gap, score, gamma_t ? gamma_t + p : nullptr);
  if (threadIdx.x == 0 && best) best[p] = b.pos >= 0 ? it.cell[beg + b.pos] : -1;
}

cudaError_t launch_prep(const Set& set, const Items& it, const Plan& pl, float* tables, uint64_t* sums,
                        cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  note_launch();
  k_prep<<<it.n * 2, kPrepThreads, 0, s>>>(set, it, pl, tables, sums);
  return cudaGetLastError();
}

static int score_lcap(const Dims& d) {
  const int lc = (d.theta_cap + 3) & ~3;
  return lc < kSmemTableCap ? lc : kSmemTableCap;
}

static int score_qwin(const Dims& d, const Plan& pl) {
  const int w = ((pl.W + 3) & ~3) + 4;
  return w < d.Q ? w : d.Q;
}

static size_t score_smem(const Dims& d, const Plan& pl) {
  return 16 + (size_t)score_qwin(d, pl) * 4 + 2 * (size_t)(kTableHeader + 3 * score_lcap(d)) * 4;
}

cudaError_t launch_score(const Set& set, const Items& it, const Plan& pl, const float* tables, uint64_t* sums,
                         void* dump, int dump_stride, int sm_count, cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  const long long tiles = (long long)it.n * pl.O * pl.chunks;
  if (tiles > 0x7fffffffLL) return cudaErrorInvalidValue;
  const size_t smem = score_smem(set.d, pl);
  const int lcap_s = score_lcap(set.d), qwin = score_qwin(set.d, pl);
  int per_sm = 0;
  cudaError_t e;
  if (dump) {
    e = cudaFuncSetAttribute(k_score<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_score<true>, kScoreThreads, smem);
  } else {
    e = cudaFuncSetAttribute(k_score<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_score<false>, kScoreThreads, smem);
  }
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  const long long cap = (long long)per_sm * sm_count;
  const int grid = (int)(tiles < cap ? tiles : cap);
  note_launch();
  if (dump)
    k_score<true><<<grid, kScoreThreads, smem, s>>>(set, it, pl, tables, sums, (unsigned char*)dump, dump_stride,
                                                    (int)tiles, lcap_s, qwin);
  else
    k_score<false><<<grid, kScoreThreads, smem, s>>>(set, it, pl, tables, sums, nullptr, 0, (int)tiles, lcap_s,
                                                     qwin);
  return cudaGetLastError();
}

cudaError_t launch_finalize(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums, double* gap,
                            double* score, float* gamma_t, int32_t* best, cudaStream_t s) {
  note_launch();
  k_finalize<<<it.off ? set.P : 1, 256, 0, s>>>(set, it, pl, sums, gap, score, gamma_t, best);
  return cudaGetLastError();
}

}  // namespace fs
