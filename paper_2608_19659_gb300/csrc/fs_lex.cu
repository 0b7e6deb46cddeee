// Tiers 3 and 4 of the lexicographic objective (Section 3) and the goodput
// gap (Fig. 4a; the third stage of Section 4.2's stage-wise gap), for sm_103a.
//
// Section 3 orders the objective: (1) critical floors, (2) max min_i r_i,
// (3) maximise total served goodput, (4) minimise fragmentation. The
// threshold solver (k_solve) settles tiers 1-2 (t*, floors met). Among the
// allocations that keep them optimal -- every class at r_i >= max(t*,
// delta_i) when t* > 0; at t* = 0 the critical classes at their floors and
// the others free; nothing at all when the floors cannot be met -- tier 3
// takes the most goodput, sum_i x_i with x_i = min(lambda_i, n c) (Eqs. 2
// and 4), each class's term in fixed point rint(x_i 2^20) so that sums are
// exact; tier 4 the fewest GPUs in use, then class by class the threshold
// solver's tie rules (no replicas first, lower TP, fewer replicas; the row's
// best bin carries the larger-capacity and lower-bin rules).
//
// For a fixed (TP, n) a larger capacity never lowers goodput or fulfilment,
// so one row per (class, TP) -- its best SLO-feasible bin -- carries every
// useful option, and replica counts past the first that serves the whole
// demand add GPUs and no goodput. The optimum is a programme over classes and
// GPUs left: S_i(g) = the best (goodput, -GPUs) of classes i..K-1 within g
// GPUs, S_K = 0, S_i(g) = max over class i's options (cost <= g) of their
// goodput plus S_{i+1}(g - cost).
//
// k_solve_lex: one CTA per realisation; the table S in global scratch,
//   threads over g, one class per step; thread 0 then walks the classes
//   forward taking the preferred option that keeps the optimum.
// k_score_goodput: the goodput stage of the Monte-Carlo score. Within a
//   segment (candidate e, outcome o) a scenario's goodput gap
//   |GP(A+') - GP(A-')| depends on its draw only through (c_y position,
//   tail gate), as its t* does: the block tabulates those values (a warp per
//   entry: each realisation's row capacity and t* as the scorer computes
//   them, then the programme over the classes with row r patched, lanes over
//   g), then draws every scenario's position and sums the entries.
// k_finalize_goodput: E[Gamma_gp,t+1 | e] = sum 2^-20 / (O S) / sum lambda,
//   the score Gamma_gp,t - E and the argmax (same order as the max-min stage).
#include <cuda_runtime.h>

#include "fs_finalize.cuh"
#include "fs_internal.cuh"
#include "fs_sample.cuh"

namespace fs {

// A class's served goodput in 2^-20 req/s: rint(min(lambda, fl(n c)) 2^20)
// (2^20 x is exact; the conversion rounds to nearest, ties to even).
__device__ __forceinline__ long long goodput_fx(float n, float c, float lam) {
  const float served = __fmul_rn(n, c);
  const float x = served < lam ? served : lam;
  return __float2ll_rn(__fmul_rn(x, 0x1p20f));
}

// One programme cell: goodput (-1: unreachable) and GPUs in use.
struct LexCell {
  long long gp;
  int gpus;
};

__device__ __forceinline__ bool lex_better(long long gpa, int gpusa, long long gpb, int gpusb) {
  return gpa > gpb || (gpa == gpb && gpusa < gpusb);
}

// --------------------------------------------------------------------------- tiers 3-4

__global__ void __launch_bounds__(256) k_solve_lex(Set set, int n_real, const float* cap_x, const float* tail_x,
                                                   fs_allocation* out_x, LexCell* scratch, int r0) {
  const Dims& d = set.d;
  const int r = r0 + blockIdx.x;
  const int tid = threadIdx.x;
  if (r >= n_real) return;
  const float* cap;
  const float* tail;
  fs_allocation* out;
  if (cap_x) {
    cap = cap_x + (size_t)r * d.cells;
    tail = tail_x + (size_t)r * d.cells;
    out = out_x + r;
  } else {
    const int p = r >> 1, sigma = r & 1;
    const float* bp = set.bounds + (size_t)p * 4 * d.cells;
    cap = bp + (size_t)(sigma ? CAP_HI : CAP_LO) * d.cells;
    tail = bp + (size_t)(sigma ? TAIL_LO : TAIL_HI) * d.cells;
    out = set.base + r;
  }
  LexCell* S = scratch + (size_t)blockIdx.x * (size_t)(d.K + 1) * (d.G + 1);
  __shared__ float sC[256];
  __shared__ int sB[256];
  __shared__ float sT[FS_MAX_CLASSES];
  __shared__ int sEmpty[FS_MAX_CLASSES];
  const float tstar = out->t_star;
  const int met = out->floors_met;
  // rows: best SLO-feasible bin (largest capacity, then lowest bin)
  for (int rho = tid; rho < d.K4; rho += blockDim.x) {
    const int i = rho >> 2;
    const float L = set.slo[i];
    float best = 0.0f;
    int bb = -1;
    for (int b = 0; b < d.B; ++b) {
      const size_t c = (size_t)rho * d.B + b;
      if (tail[c] <= L) {
        const float v = __fadd_rn(cap[c], 0.0f);  // -0 as +0
        if (bb < 0 || v > best) {
          best = v;
          bb = b;
        }
      }
    }
    sC[rho] = best;
    sB[rho] = bb;
  }
  for (int i = tid; i < d.K; i += blockDim.x) {
    const float dl = set.slo[d.K + i];  // floors follow the SLOs (0: not critical)
    sT[i] = tstar > 0.0f ? fmaxf(tstar, dl) : dl;
    sEmpty[i] = !(tstar > 0.0f) && !(dl > 0.0f);
  }
  if (!met) {  // tier 1 cannot hold: nothing is allocated (k_solve wrote the empty allocation)
    if (tid == 0) out->goodput = 0.0;
    return;
  }
  for (int g = tid; g <= d.G; g += blockDim.x) S[(size_t)d.K * (d.G + 1) + g] = LexCell{0, 0};
  __syncthreads();
  for (int i = d.K - 1; i >= 0; --i) {
    const LexCell* nxt = S + (size_t)(i + 1) * (d.G + 1);
    LexCell* cur = S + (size_t)i * (d.G + 1);
    const float lam = set.lam[i], T = sT[i];
    for (int g = tid; g <= d.G; g += blockDim.x) {
      LexCell best{-1, 0};
      if (sEmpty[i] && nxt[g].gp >= 0) best = nxt[g];
      for (int j = 0; j < kT; ++j) {
        if (sB[4 * i + j] < 0) continue;
        const float C = sC[4 * i + j];
        const int M = rep_cap(d, j);
        for (int n = 1; n <= M && (n << j) <= g; ++n) {
          const float nf = (float)n;
          if (T > 0.0f && !(fulfil(nf, C, lam) >= T)) continue;
          const LexCell pv = nxt[g - (n << j)];
          if (pv.gp >= 0) {
            const long long v = goodput_fx(nf, C, lam) + pv.gp;
            const int u = (n << j) + pv.gpus;
            if (best.gp < 0 || lex_better(v, u, best.gp, best.gpus)) best = LexCell{v, u};
          }
          if (!(__fmul_rn(nf, C) < lam)) break;  // the whole demand served: more replicas add nothing
        }
      }
      cur[g] = best;
    }
    __syncthreads();
  }
  if (tid != 0) return;
  // forward: class by class the preferred option that keeps the optimum
  int left = d.G, total = 0;
  const long long gp_all = S[d.G].gp;
  for (int i = 0; i < d.K; ++i) {
    const LexCell target = S[(size_t)i * (d.G + 1) + left];
    const LexCell* nxt = S + (size_t)(i + 1) * (d.G + 1);
    const float lam = set.lam[i], T = sT[i];
    int cj = -1, cn = 0;
    if (!(sEmpty[i] && nxt[left].gp == target.gp && nxt[left].gpus == target.gpus)) {
      for (int j = 0; j < kT && cj < 0; ++j) {
        if (sB[4 * i + j] < 0) continue;
        const float C = sC[4 * i + j];
        const int M = rep_cap(d, j);
        for (int n = 1; n <= M && (n << j) <= left; ++n) {
          const float nf = (float)n;
          if (T > 0.0f && !(fulfil(nf, C, lam) >= T)) continue;
          const LexCell pv = nxt[left - (n << j)];
          if (pv.gp >= 0 && goodput_fx(nf, C, lam) + pv.gp == target.gp && (n << j) + pv.gpus == target.gpus) {
            cj = j;
            cn = n;
            break;
          }
        }
      }
    }
    out->tp[i] = (int8_t)(cj >= 0 ? 1 << cj : 0);
    out->bin[i] = (int16_t)(cj >= 0 ? sB[4 * i + cj] : -1);
    out->replicas[i] = (int16_t)cn;
    out->fulfil[i] = cj >= 0 ? fulfil((float)cn, sC[4 * i + cj], lam) : 0.0f;
    if (cj >= 0) {
      left -= cn << cj;
      total += cn << cj;
    }
  }
  out->total_gpus = total;
  out->goodput = (double)gp_all * 0x1p-20;
}

// --------------------------------------------------------------------------- goodput stage

// rint(min(lambda, fl(n c)) 2^20), the same value as goodput_fx, for
// 0 <= min(...) <= 2^20 (the host requires sum lambda <= 2^20): x 2^-20 is
// exact there (or its rint is 0 either way), and fixed40 rounds its 2^40
// multiple to nearest, ties to even, without a float-to-int64 conversion.
__device__ __forceinline__ long long goodput_fx20(float n, float c, float lam) {
  const float served = __fmul_rn(n, c);
  const float x = served < lam ? served : lam;
  return (long long)fixed40(__fmul_rn(x, 0x1p-20f));
}

// The options of one row in a realisation: replica counts [lo, hi] (lo = 0:
// none) at capacity C, and the thresholds T in (a, b] for which they stay so.
struct RowOpt {
  float C;
  int lo, hi;
  float a, b;
};

// Class i's options on row (i, tau = 2^j) at capacity C are the replica
// counts n in [1, M = G / tau] whose fulfilment reaches T (all of them when
// T = 0), up to the first that serves the whole demand (fl(n C) >= lambda:
// more replicas add GPUs and no goodput). Both ends are monotone in n, so the
// options are one range [lo, hi]: the smallest feasible count by
// min_replicas, the first saturating count by bisection. lo = 0: none.
__device__ __forceinline__ void row_range(float C, bool ok, int M, float T, float lam, float rl, int& lo, int& hi) {
  lo = hi = 0;
  if (!ok || M < 1) return;
  lo = T > 0.0f ? min_replicas(T, C, lam, rl, (float)M) : 1;
  if (lo == 0) return;
  int a = 1, b = M + 1;  // the first n in [1, M] with fl(n C) >= lambda, else M + 1
  while (a < b) {
    const int mid = (a + b) >> 1;
    if (!(__fmul_rn((float)mid, C) < lam)) b = mid;
    else a = mid + 1;
  }
  hi = min(M, max(lo, a));
}

// The row's range and the interval of thresholds that gives the same lo (and
// so the same hi): fulfil(lo - 1) < T <= fulfil(lo) for lo >= 1 (no lower end
// at lo = 1), T > fulfil(M) for lo = 0 (fulfil is nondecreasing in n).
__device__ __forceinline__ RowOpt row_opt(float C, bool ok, int M, float T, float lam, float rl) {
  RowOpt r{C, 0, 0, -INFINITY, INFINITY};
  row_range(C, ok, M, T, lam, rl, r.lo, r.hi);
  if (!ok || M < 1) return r;
  if (r.lo == 0) {
    r.a = fulfil((float)M, C, lam);
  } else {
    r.b = fulfil((float)r.lo, C, lam);
    if (r.lo > 1) r.a = fulfil((float)(r.lo - 1), C, lam);
  }
  return r;
}

__device__ __forceinline__ float class_threshold(float t, float dl) { return t > 0.0f ? fmaxf(t, dl) : dl; }

// The best tier-3 goodput of every class but `skip` within g GPUs, for g in
// [0, G], at tiers 1-2 value t (-1: the floors of those classes cannot be
// met within g), by one warp: the programme over the classes (no replicas,
// when class i may stay empty: T_i = 0 and no floor; else one range of
// replica counts on each of its rows) with lanes over g. Also leaves in opt
// every row's range at t (those of `skip` for warp_best_with; row `fixed`,
// whose capacity varies, with no interval). dpa, dpb: the warp's two arrays
// of G + 1 cells. Returns the array that holds the result.
template <bool FL>
__device__ const long long* warp_other(const Dims& d, const float* sCs, const int* sOk, const float* sLam,
                                       const float* sRl, const float* sDl, int skip, int fixed, float t,
                                       RowOpt* opt, long long* dpa, long long* dpb) {
  const int lane = threadIdx.x & 31;
  __syncwarp();  // the previous result and ranges are no longer read
  for (int rho = lane; rho < d.K4; rho += 32) {
    const int i = rho >> 2;
    RowOpt r = row_opt(sCs[rho], sOk[rho] != 0, d.G >> (rho & 3), class_threshold(t, FL ? sDl[i] : 0.0f),
                       sLam[i], sRl[i]);
    if (rho == fixed) r.a = -INFINITY, r.b = INFINITY;
    opt[rho] = r;
  }
  for (int g = lane; g <= d.G; g += 32) dpa[g] = 0;
  __syncwarp();
  long long* cur = dpa;  // S_{i+1}
  long long* nxt = dpb;
  for (int i = d.K - 1; i >= 0; --i) {
    if (i == skip) continue;
    const float dl = FL ? sDl[i] : 0.0f;
    const bool may_empty = !(t > 0.0f) && !(dl > 0.0f);
    const float lam = sLam[i];
    for (int g = lane; g <= d.G; g += 32) {
      long long best = may_empty ? cur[g] : -1;
#pragma unroll
      for (int j = 0; j < kT; ++j) {
        const RowOpt ro = opt[4 * i + j];
        const int top = min(ro.hi, g >> j);
        for (int n = ro.lo; n <= top && n > 0; ++n) {
          const long long pv = cur[g - (n << j)];
          if (pv >= 0) {
            const long long v = goodput_fx20((float)n, ro.C, lam) + pv;
            best = v > best ? v : best;
          }
        }
      }
      nxt[g] = best;
    }
    __syncwarp();
    long long* x = cur;
    cur = nxt;
    nxt = x;
  }
  return cur;
}

// Whether the ranges in opt (left by warp_other at a value t0 with
// (t0 > 0) = pos) hold at t as well: then so do the programme's result and
// class i_r's other rows. One warp.
template <bool FL>
__device__ bool warp_ranges_hold(const Dims& d, const float* sDl, const RowOpt* opt, float t, bool pos) {
  const int lane = threadIdx.x & 31;
  bool ok = (t > 0.0f) == pos;
  for (int rho = lane; rho < d.K4; rho += 32) {
    const float T = class_threshold(t, FL ? sDl[rho >> 2] : 0.0f);
    ok = ok && opt[rho].a < T && T <= opt[rho].b;
  }
  return __all_sync(0xffffffffu, ok);
}

// Tier-3 goodput of one realisation with row rr at capacity Cr (its range
// [lor, hir] at t), at tiers 1-2 value t, given other = warp_other(..., skip
// = class of rr, t): the best over class i_r's choices (nothing, when it may
// stay empty; else n replicas on one of its rows) of its goodput plus the
// others' best within the GPUs left; -1 when the floors cannot be met. Lanes
// over the choices, one warp.
template <bool FL>
__device__ long long warp_best_with(const Dims& d, const float* sLam, const float* sDl, const RowOpt* opt, int rr,
                                    float Cr, int lor, int hir, float t, const long long* other) {
  const int lane = threadIdx.x & 31, ir = rr >> 2, jr = rr & 3;
  const float lam = sLam[ir];
  const float dl = FL ? sDl[ir] : 0.0f;
  int cnt[kT], lo[kT];
  float C[kT];
#pragma unroll
  for (int j = 0; j < kT; ++j) {
    const RowOpt ro = opt[4 * ir + j];
    lo[j] = j == jr ? lor : ro.lo;
    const int hi = j == jr ? hir : ro.hi;
    C[j] = j == jr ? Cr : ro.C;
    cnt[j] = lo[j] > 0 ? hi - lo[j] + 1 : 0;
  }
  long long best = (!(t > 0.0f) && !(dl > 0.0f)) ? other[d.G] : -1;
  const int e1 = cnt[0], e2 = e1 + cnt[1], e3 = e2 + cnt[2], total = e3 + cnt[3];
  for (int x = lane; x < total; x += 32) {
    int j, n;
    float Cj;
    if (x < e1) { j = 0; n = lo[0] + x; Cj = C[0]; }
    else if (x < e2) { j = 1; n = lo[1] + (x - e1); Cj = C[1]; }
    else if (x < e3) { j = 2; n = lo[2] + (x - e2); Cj = C[2]; }
    else { j = 3; n = lo[3] + (x - e3); Cj = C[3]; }
    const long long pv = other[d.G - (n << j)];
    if (pv >= 0) {
      const long long v = goodput_fx20((float)n, Cj, lam) + pv;
      best = v > best ? v : best;
    }
  }
  for (int off = 16; off; off >>= 1) {
    const long long o = __shfl_xor_sync(0xffffffffu, best, off);
    best = o > best ? o : best;
  }
  return best;
}

// t* of realisation sigma at row capacity C, from the candidate's table in
// global memory (the IEEE row term: every input).
template <bool FL>
__device__ __forceinline__ float tstar_global(const float* h, float C) {
  const int Lp = __float_as_int(h[H_LPAD]);
  const float* kap = h + kTableHeader;
  const float* thx = kap + Lp;
  const float* mnx = thx + Lp;
  int pos = 0;
  for (int step = __float_as_int(h[H_STEP0]); step > 0; step >>= 1) pos += kap[pos + step - 1] <= C ? step : 0;
  const float thb = thx[pos];
  const float m = mnx[pos];
  const float tr = m >= 1.0f ? fulfil(m, C, h[H_LAM]) : 0.0f;
  if (FL) return (tr > thb && tr >= h[H_DLT]) ? tr : thb;
  return tr > thb ? tr : thb;
}

// Shared memory of k_score_goodput: per table entry its gap (8 bytes), both
// realisations' row capacities (8) and values (16: t*, then the goodput),
// one flag byte; per warp its K4 row ranges and two programme arrays.
struct GoodputSmem {
  size_t gtab, cap, val, flag, warps, per_warp, total;
};

__host__ __device__ inline GoodputSmem goodput_smem(int K4, int G, int gt_len, int nwarp) {
  GoodputSmem m{};
  auto up = [](size_t x) { return (x + 15) & ~(size_t)15; };
  m.gtab = 0;
  m.cap = up(m.gtab + 8 * (size_t)gt_len);
  m.val = up(m.cap + 8 * (size_t)gt_len);
  m.flag = up(m.val + 16 * (size_t)gt_len);
  m.warps = up(m.flag + (size_t)gt_len);
  m.per_warp = up(sizeof(RowOpt) * (size_t)K4) + 16 * ((size_t)G + 1);
  m.total = m.warps + (size_t)nwarp * m.per_warp;
  return m;
}

// One block per segment (candidate e, outcome o) at a time. Entries: [0, W)
// open gate at position k; [W, 2W) closed gate at position k - W (under the
// prior), or W alone (closed, one value). A realisation's goodput depends on
// an entry only through its patched row capacity C' (t* is a function of
// C'), and consecutive entries often share C' (every position whose c_y lies
// at or below Cexcl, or is clamped by the refit): a run of equal C' takes one
// evaluation. The evaluation splits the programme at class i_r: the other
// classes' best within g GPUs depends on the entry only through the replica
// ranges that t* leaves their rows, which change at few values of t* in a
// segment, so a warp reruns that part only where a range changes and
// otherwise only combines it with class i_r's choices. Then the same draws
// and sums as the table path.
// MINB: resident blocks per SM the registers are capped for (2, or 4 for
// launches of many segments, whose throughput gains more from the occupancy
// than each block loses).
template <bool FL, bool RF, int MINB>
__global__ void __launch_bounds__(256, MINB) k_score_goodput(Set set, Items it, Plan pl, const float* rec,
                                                          uint64_t* sums) {
  extern __shared__ __align__(16) unsigned char smraw[];
  const Dims& d = set.d;
  const int W = pl.W, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const int gt_len = RF ? 2 * W : W + 1;
  const GoodputSmem lay = goodput_smem(d.K4, d.G, gt_len, nwarp);
  uint64_t* gtab = reinterpret_cast<uint64_t*>(smraw + lay.gtab);
  float* cap = reinterpret_cast<float*>(smraw + lay.cap);          // [2][gt_len]
  long long* val = reinterpret_cast<long long*>(smraw + lay.val);  // [2][gt_len]
  uint8_t* flag = smraw + lay.flag;  // bit 0 / 1: a run starts here (realisation 0 / 1); bit 2: reachable
  unsigned char* wbase = smraw + lay.warps + (size_t)warp * lay.per_warp;
  RowOpt* opt = reinterpret_cast<RowOpt*>(wbase);
  long long* dpa = reinterpret_cast<long long*>(wbase + ((sizeof(RowOpt) * (size_t)d.K4 + 15) & ~(size_t)15));
  long long* dpb = dpa + (d.G + 1);
  __shared__ float sC[2][256];
  __shared__ int sOk[2][256];
  __shared__ float sLam[FS_MAX_CLASSES], sRl[FS_MAX_CLASSES], sDl[FS_MAX_CLASSES];
  for (int x = tid; x < 2 * d.K4; x += blockDim.x) {
    const int sg = x / d.K4, rho = x - sg * d.K4;
    sC[sg][rho] = set.rowC[(size_t)sg * d.K4 + rho];
    sOk[sg][rho] = set.rowB[(size_t)sg * d.K4 + rho] >= 0;
  }
  for (int i = tid; i < d.K; i += blockDim.x) {
    sLam[i] = set.lam[i];
    sRl[i] = __frcp_rn(set.lam[i]);
    sDl[i] = FL ? set.slo[d.K + i] : 0.0f;
  }
  __syncthreads();
  const PhiloxKeys keys{};  // (the plan's round keys serve a one-problem launch)
  const long long n_seg = (long long)it.n * pl.O;
  for (long long seg = blockIdx.x; seg < n_seg; seg += gridDim.x) {
    const long long* other = nullptr;  // the warp's programme over the other classes, for this segment
    bool other_pos = false;
    int other_sg = 0;
    const int item = (int)(seg / pl.O), o = (int)(seg - (long long)item * pl.O);
    const float* r = rec + (size_t)item * pl.item_floats;
    const float* h0 = r;
    const float* h1 = r + d.slot_floats;
    const float* win = r + 2 * (size_t)d.slot_floats + (size_t)o * pl.Wp;
    const int cell = __float_as_int(h0[H_CELL]);
    if (cell < 0 || cell >= d.cells) continue;  // flagged by the preparation (uniform over the block)
    const int rr = cell / d.B;
    const uint32_t kgs = (uint32_t)__float_as_int(win[0]) << pl.sh;
    const uint32_t kgs16 = (uint32_t)min((unsigned long long)kgs << 16, 0xFFFFFFFFull);
    const bool any_open = kgs != 0u, any_closed = kgs16 != 0xFFFFFFFFu;
    const RowCap a0 = row_cap_of(h0), a1 = row_cap_of(h1);
    auto reachable = [&](int k) { return k < W ? any_open : any_closed; };
    // each entry's patched row capacity in both realisations
    for (int k = tid; k < gt_len; k += blockDim.x) {
      const bool g = k < W;
      const float cy = g ? win[4 + k] : (RF ? win[4 + k - W] : 0.0f);
      cap[k] = RF ? row_cap(a0, cy, g) : (g ? fmaxf(a0.pc, cy) : a0.pc);
      cap[gt_len + k] = RF ? row_cap(a1, cy, g) : (g ? fmaxf(a1.pc, cy) : a1.pc);
    }
    __syncthreads();
    // where runs of equal capacity start, and t* there
    for (int k = tid; k < gt_len; k += blockDim.x) {
      uint8_t f = 0;
      if (reachable(k)) {
        f = 4;
        const bool first = k == 0 || !reachable(k - 1);
        const float c0 = cap[k], c1 = cap[gt_len + k];
        if (first || __float_as_uint(c0) != __float_as_uint(cap[k - 1])) {
          f |= 1;
          val[k] = (long long)__float_as_uint(tstar_global<FL>(h0, c0));
        }
        if (first || __float_as_uint(c1) != __float_as_uint(cap[gt_len + k - 1])) {
          f |= 2;
          val[gt_len + k] = (long long)__float_as_uint(tstar_global<FL>(h1, c1));
        }
      }
      flag[k] = f;
    }
    __syncthreads();
    // the warps take chunks of 32 entries of one realisation in turn; a chunk's
    // first reachable entry starts a run. Every run start's row-r range comes
    // from its own lane; the others' programme is rerun only where a row's
    // range changes with t*
    {
      const int ir = rr >> 2, jr = rr & 3;
      const float lam_r = sLam[ir], rl_r = sRl[ir], dl_r = FL ? sDl[ir] : 0.0f;
      const int n_chunk = (gt_len + 31) >> 5;
      for (int task = warp; task < 2 * n_chunk; task += nwarp) {
        const int sg = task & 1, kk = ((task >> 1) << 5) + lane;
        const float* cs = cap + (size_t)sg * gt_len;
        long long* v = val + (size_t)sg * gt_len;
        const bool reach = kk < gt_len && (flag[kk] & 4);
        const bool start = reach && ((flag[kk] >> sg) & 1);
        const unsigned rb = __ballot_sync(0xffffffffu, reach);
        const bool head = start || (rb && lane == __ffs(rb) - 1);
        float c = 0.0f, t = 0.0f;
        int lor = 0, hir = 0;
        if (head) {  // t* stored where a run starts, else evaluated
          c = cs[kk];
          t = start ? __uint_as_float((uint32_t)v[kk]) : tstar_global<FL>(sg ? h1 : h0, c);
          row_range(c, true, d.G >> jr, class_threshold(t, dl_r), lam_r, rl_r, lor, hir);
        }
        unsigned heads = __ballot_sync(0xffffffffu, head);
        long long mine = 0;
        while (heads) {
          const int p = __ffs(heads) - 1;
          heads &= heads - 1;
          const float tp = __shfl_sync(0xffffffffu, t, p), cp = __shfl_sync(0xffffffffu, c, p);
          const int lop = __shfl_sync(0xffffffffu, lor, p), hip = __shfl_sync(0xffffffffu, hir, p);
          if (other == nullptr || other_sg != sg || !warp_ranges_hold<FL>(d, sDl, opt, tp, other_pos)) {
            other = warp_other<FL>(d, sC[sg], sOk[sg], sLam, sRl, sDl, ir, rr, tp, opt, dpa, dpb);
            other_pos = tp > 0.0f;
            other_sg = sg;
          }
          long long gv = warp_best_with<FL>(d, sLam, sDl, opt, rr, cp, lop, hip, tp, other);
          gv = gv < 0 ? 0 : gv;
          if (lane >= p) mine = gv;
        }
        if (reach) v[kk] = mine;
      }
    }
    __syncthreads();
    for (int k = tid; k < gt_len; k += blockDim.x) {
      if (!(flag[k] & 4)) continue;
      const long long g0 = val[k], g1 = val[gt_len + k];
      const unsigned long long gap = (unsigned long long)(g1 > g0 ? g1 - g0 : g0 - g1);
      gtab[k] = gap;
    }
    __syncthreads();
    unsigned long long v = sample_gtab<true, RF>(pl, keys, o, cell, 0, pl.calls, smem_u32(gtab), kgs16);
    for (int off = 16; off; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    if (lane == 0 && v) atomicAdd(reinterpret_cast<unsigned long long*>(&sums[(size_t)seg]), v);
    __syncthreads();  // the tables are rebuilt for the next segment
  }
}

// E, score and argmax of the goodput stage for one problem (one CTA).
__global__ void k_finalize_goodput(Set set, Items it, Plan pl, const uint64_t* sums, double lam_sum, double* gap,
                                   double* score, double* gamma, int32_t* best, uint32_t* status_copy) {
  __shared__ Best sb[32];
  // every earlier kernel of the call has completed: the status word travels
  // with the outputs
  if (threadIdx.x == 0 && status_copy) *status_copy = *set.status;
  const Dims& d = set.d;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarp = blockDim.x >> 5;
  const long long gm = __double2ll_rn(__dmul_rn(set.base[0].goodput, 0x1p20));
  const long long gpl = __double2ll_rn(__dmul_rn(set.base[1].goodput, 0x1p20));
  const long long gfix = gpl > gm ? gpl - gm : gm - gpl;
  const long long n = (long long)pl.O * pl.S;
  const double dn = __ll2double_rn(n);
  Best b = no_best();
  for (int q = tid; q < it.n; q += blockDim.x) {
    const int cell = it.cell[q];
    long long tot = 0;
    for (int o = 0; o < pl.O; ++o) tot += (long long)sums[(size_t)q * pl.O + o];
    const long long sc = gfix * n - tot;
    if (gap) gap[q] = __ddiv_rn(__ddiv_rn(__dmul_rn(__ll2double_rn(tot), 0x1p-20), dn), lam_sum);
    if (score) score[q] = __ddiv_rn(__ddiv_rn(__dmul_rn(__ll2double_rn(sc), 0x1p-20), dn), lam_sum);
    const Best c = make_best(sc, (cell / d.B) & 3, q, cell);
    if (better(c, b)) b = c;
  }
  b = warp_best(b);
  if (lane == 0) sb[warp] = b;
  __syncthreads();
  if (warp == 0) {
    b = warp_best(lane < nwarp ? sb[lane] : no_best());
    if (lane == 0) {
      if (best) *best = b.valid() ? b.cell : -1;
      if (gamma) *gamma = __ddiv_rn(__dmul_rn(__ll2double_rn(gfix), 0x1p-20), lam_sum);
    }
  }
}

// --------------------------------------------------------------------------- launchers

size_t lex_scratch_cells(const Dims& d) { return (size_t)(d.K + 1) * (d.G + 1); }

cudaError_t launch_solve_lex(const Set& set, int n, const float* cap_x, const float* tail_x, fs_allocation* out,
                             void* scratch, int per_launch, cudaStream_t s) {
  for (int r0 = 0; r0 < n; r0 += per_launch) {
    const int m = n - r0 < per_launch ? n - r0 : per_launch;
    note_launch();
    k_solve_lex<<<m, 256, 0, s>>>(set, n, cap_x, tail_x, out, static_cast<LexCell*>(scratch), r0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

int goodput_threads(const Dims& d, const Plan& pl, bool rf, size_t* smem) {
  const int gt_len = rf ? 2 * pl.W : pl.W + 1;
  for (int nw = 8; nw >= 1; --nw) {
    const GoodputSmem m = goodput_smem(d.K4, d.G, gt_len, nw);
    if (m.total <= kGoodputSmemMax) {
      if (smem) *smem = m.total;
      return 32 * nw;
    }
  }
  return 0;
}

cudaError_t launch_score_goodput(const Set& set, const Items& it, const Plan& pl, const float* tables,
                                 uint64_t* sums, int floors, int sm_count, cudaStream_t s) {
  if (it.n <= 0) return cudaSuccess;
  const bool rf = set.prior == 1;
  size_t smem = 0;
  const int threads = goodput_threads(set.d, pl, rf, &smem);
  if (threads == 0) return cudaErrorInvalidValue;  // refused by the host before this point
  // many segments (beyond four waves of two blocks per SM): the instance with
  // registers for four blocks per SM (measured 5.94 -> 3.44 ms on the
  // eight-class workload, 0.375 -> 0.325 ms on the mid one at three times its
  // demands; the paper-scale call, one wave, slower: 0.17 -> 0.19 ms)
  const long long n_seg = (long long)it.n * pl.O;
  const bool wide = n_seg > 4LL * 2 * sm_count;
#define FS_GP(MB) \
  (floors ? (rf ? k_score_goodput<true, true, MB> : k_score_goodput<true, false, MB>) \
          : (rf ? k_score_goodput<false, true, MB> : k_score_goodput<false, false, MB>))
  auto kern = wide ? FS_GP(4) : FS_GP(2);
#undef FS_GP
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(kern), smem);
  if (e != cudaSuccess) return e;
  // one block per segment: segments differ widely in cost (where row r sets
  // t*, its ranges change often), and the block scheduler evens them out
  const long long grid = n_seg < 0x7fffffffLL ? n_seg : 0x7fffffffLL;
  note_launch();
  kern<<<(unsigned)grid, threads, smem, s>>>(set, it, pl, tables, sums);
  return cudaGetLastError();
}

cudaError_t launch_finalize_goodput(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                                    double lam_sum, double* gap, double* score, double* gamma, int32_t* best,
                                    uint32_t* status_copy, cudaStream_t s) {
  note_launch();
  k_finalize_goodput<<<1, 256, 0, s>>>(set, it, pl, sums, lam_sum, gap, score, gamma, best, status_copy);
  return cudaGetLastError();
}

}  // namespace fs
