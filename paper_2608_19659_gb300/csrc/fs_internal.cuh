// Internal device-side definitions of the decision-gap scorer (sm_103a).
//
// Layout of a problem set in HBM (all problems share K, B, G, SLOs, demands
// and the quantile table; the replay batches one problem per reveal order):
//   bounds   [P][4][cells] f32   rows CAP_LO, CAP_HI, TAIL_LO, TAIL_HI
//   revealed [P][cells]    u8
//   theta    [P][2][theta_cap] f32  sorted option fulfilments of the base
//                                   realisation sigma (0 = A-, 1 = A+)
//   ntheta   [P][2]        i32
//   rowC     [P][2][K*4]   f32   best SLO-feasible capacity per (class, TP)
//   rowB     [P][2][K*4]   i32   its bin (-1: none)
//   base     [P][2]        fs_allocation
//   work     [4]           u64   chunk counter of the Monte-Carlo kernel, the reduction's ticket,
//                                 table entries evaluated and scenarios that tested their tail
//                                 gate (both accumulate across calls; the host zeroes them)
// Per scoring call (items = (problem, candidate cell) pairs), one record of
// item_floats = 2 slot_floats + O Wp floats per item:
//   [2][slot_floats] f32   threshold tables of the two realisations
//   [O][Wp]          f32   per outcome: the gate position (int) and three pad
//                          words, then the outcome's W quantiles mapped into the
//                          candidate's capacity interval (Wp = 4 + W rounded up to 4)
//   sums     [items][O]    u64 (int64 fixed point, 2^-40)
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/fleetsieve.h"

namespace fs {

constexpr int kT = 4;                 // TP degrees {1, 2, 4, 8}
constexpr int kCostInf = 0x3FFFFFFF;  // "no option covers the threshold"
constexpr int kSolveThreads = 256;
constexpr int kSolveThreadsWide = 512;  // a scoring solve of a model with more than 256 cells
constexpr int kPrepThreads = 256;
constexpr int kScoreThreads = 256;
constexpr int kTableHeader = 20;      // floats before the three table arrays (16-byte multiple)
constexpr int kSmemTableCap = 256;    // table entries staged in shared memory per realisation (pow2)
// Row table of a scoring solve: one word per (row, threshold) pair, built when
// K4 x |Theta| is at most this (else the per-candidate preparation searches).
constexpr int kRowTabMax = 8192;

// Table header words (floats unless noted).
enum : int {
  H_TH_BASE = 0,  // threshold below the first table entry (0 if none)
  H_TCL = 1,      // t* of this realisation at row capacity Cexcl: every scenario whose tail gate is closed
  H_L = 2,        // entries (int)
  H_LPAD = 3,     // entries padded to 4 (int)
  // Row r's capacity C' in a scenario drawing c_y with tail gate g (Eq. 5):
  //   C' = max(g ? max(P_open, c_y) : P_closed, min(max(c_y, F_lo), F_hi))
  // Without the structural prior P_open = P_closed = Cexcl (the row's best
  // SLO-feasible capacity without the candidate's bin) and F_lo = F_hi = 0;
  // with it the row's other bins are refit by the draw (see k_prep).
  H_CX = 4,       // P_closed
  H_BX = 5,       // bin of Cexcl (int, -1 none; without the prior)
  H_PO = 6,       // P_open
  H_LAM = 7,      // demand of the candidate's class
  H_LF = 8, H_HF = 9,  // F_lo, F_hi
  H_LO_L = 10, H_HI_L = 11,  // candidate cell's tail bounds
  H_SLO = 12,     // SLO of the candidate's class
  H_CELL = 13,    // candidate cell (int)
  H_P = 14,       // problem (int)
  H_STEP0 = 15,   // first step of the table search, P/2 with P = pow2 >= L + 1 (int, 0 if L = 0)
  H_ROW = 16,     // 1 if row r can buy a replica at some reachable threshold (int)
  H_FAST = 17,    // 1 if every reachable row-term quotient is in Markstein's range (int)
  H_RLAM = 18,    // RN(1 / lambda)
  H_DLT = 19,     // floor delta of the candidate's class (0: not critical)
};

enum : int { CAP_LO = 0, CAP_HI = 1, TAIL_LO = 2, TAIL_HI = 3 };

// status word bits (device -> host)
enum : uint32_t {
  ST_TIMEOUT = 1u,       // a bounded mbarrier wait gave up
  ST_THETA = 2u,         // threshold count above the model's capacity
  ST_TABLE = 4u,         // candidate table longer than its slot
  ST_CELL = 8u,          // a device-side candidate id outside [0, cells)
};

struct Dims {
  int K, B, G, Q, cells, K4;
  int theta_cap;        // K * sum_j floor(G / tau_j): most thresholds one realisation can have
  int slot_floats;      // stride of one (item, sigma) table
  int lcap;             // table entries a slot can hold: pow2 >= theta_cap + 1, at least 4
};

struct Set {
  Dims d;
  int P;
  const float* lam;     // [K]
  const float* slo;     // [2K]: SLOs, then the critical floors delta_i (0: not critical);
                        // kernel instances without floors never read the second half
  const float* qn;      // [Q]
  float* bounds;        // [P][4][cells]
  uint8_t* revealed;    // [P][cells]
  float* theta;         // [P][2][theta_cap]
  int* ntheta;          // [P][2]
  float* rowC;          // [P][2][K4]
  int* rowB;            // [P][2][K4] bin of rowC, -1 = no SLO-feasible bin
  fs_allocation* base;  // [P][2]
  uint32_t* status;
  unsigned long long* work;  // [4] chunk counter, reduction ticket (zeroed by k_prep); table entries
                             // evaluated and scenarios that tested their tail gate in the Monte-Carlo
                             // kernel (summed over calls, zeroed by the host)
  const int* skip;      // [P] or nullptr: base solves skip problems with skip[p] >= 0
  int* rtab;            // [P][2][kRowTabMax] or nullptr: row tables of the scoring solves,
                        // word (row rho, threshold k) at k K4 + rho
  int prior;            // interval refit after a measurement: 0 the measured cell only,
                        // 1 also its row's other bins (capacity and tail nondecreasing in load)
};

// The refit of one bound after a measurement v under the monotone prior: a
// lower bound rises to v, an upper bound falls to v, clamped into [lo, hi]
// so that the interval never empties.
__host__ __device__ __forceinline__ float raise_lo(float lo, float hi, float v) { return fminf(fmaxf(lo, v), hi); }
__host__ __device__ __forceinline__ float lower_hi(float lo, float hi, float v) { return fmaxf(fminf(hi, v), lo); }

// Collapse cell to the measurement (c, l) in the bounds [4][cells] and, under
// the monotone prior, refit its row: bins above it in load get lower bounds of
// (c, l), bins below it upper bounds.
__host__ __device__ __forceinline__ void refit_cell(float* bp, int cells, int B, int prior, int cell, float c,
                                                    float l) {
  bp[0 * (size_t)cells + cell] = c;
  bp[1 * (size_t)cells + cell] = c;
  bp[2 * (size_t)cells + cell] = l;
  bp[3 * (size_t)cells + cell] = l;
  if (prior != 1) return;
  const int first = cell - cell % B, be = cell % B;
  for (int b = 0; b < B; ++b) {
    const size_t x = (size_t)first + b;
    float* clo = bp + x;
    float* chi = bp + (size_t)cells + x;
    float* tlo = bp + 2 * (size_t)cells + x;
    float* thi = bp + 3 * (size_t)cells + x;
    if (b > be) {
      *clo = raise_lo(*clo, *chi, c);
      *tlo = raise_lo(*tlo, *thi, l);
    } else if (b < be) {
      *chi = lower_hi(*clo, *chi, c);
      *thi = lower_hi(*tlo, *thi, l);
    }
  }
}

// Scenario plan shared by a launch.
struct Plan {
  uint32_t key0;        // low word of the seed
  uint32_t key1;        // high word of the seed (stream id XORed per problem)
  uint32_t stream_base; // stream id of problem 0 (problem p uses stream_base + p)
  uint32_t round;
  int O, S, W, w;       // W = Q / O quantiles per stratum, w = log2(W) <= 16
  int logO;             // log2(O) (O is a power of two)
  int sh;               // 16 - w: a 16-bit field's top w bits are field >> sh
  int calls;            // ceil(S / 4) Philox calls per (candidate, outcome)
  int Wp;               // floats per mapped outcome window: 4 + W rounded up to 4
  long long item_floats;  // floats per item record: 2 slot_floats + O Wp
  // Philox round keys of problem 0 (key1 XOR stream_base): as kernel
  // parameters at fixed offsets they are constant operands of the rounds'
  // XORs and take no registers (launches over one problem use them)
  uint32_t rk0[10], rk1[10];
  // 65536 and 8, read from the parameters rather than known to the compiler,
  // so that a word's low half moved to the top and an entry's byte offset are
  // integer multiply-adds (FMA pipe) rather than shifts and masks (ALU pipe)
  uint32_t lo16_mul, entry_bytes;
  // 0: the entry stride of a table whose entries are all equal (stored once).
  // A parameter like the others: every scenario still computes its position
  // and its entry's address, and the kernel is not specialised for that table
  uint32_t uniform_stride;
};

// Round keys of problem 0 for the plan (host).
inline void plan_round_keys(Plan& pl) {
  uint32_t k0 = pl.key0, k1 = pl.key1 ^ pl.stream_base;
  for (int r = 0; r < 10; ++r) {
    pl.rk0[r] = k0;
    pl.rk1[r] = k1;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  pl.lo16_mul = 65536u;
  pl.entry_bytes = 8u;
  pl.uniform_stride = 0u;
}

struct Items {
  int n;
  const int* p;         // [n] problem of the item, nullptr = all problem 0
  const int* cell;      // [n] candidate cell
  const int* off;       // [P + 1] item range of each problem (grouped by problem)
};

// ---------------------------------------------------------------- arithmetic

// x / lam, correctly rounded to nearest even, by Markstein's method
// (P. Markstein, "Computation of elementary functions on the IBM RISC
// System/6000 processor", IBM J. Res. Dev. 34(1), 1990): with r = RN(1/lam),
// q0 = RN(x r) is within one unit in the last place of x / lam, the residual
// x - lam q0 is exact in one fused multiply-add, and RN(q0 + (x - lam q0) r)
// is the correctly rounded quotient, provided no step overflows or underflows.
// Callers keep x in {0} or [2^-60, 2^60] and lam in [2^-60, 2^60]. Three inline
// operations instead of the out-of-line IEEE divide, so independent divisions
// overlap; the results are the IEEE quotients bit for bit.
__device__ __forceinline__ float div_markstein(float x, float lam, float rlam) {
  const float q0 = __fmul_rn(x, rlam);
  const float e = __fmaf_rn(-lam, q0, x);
  return __fmaf_rn(e, rlam, q0);
}

__device__ __forceinline__ bool in_markstein_range(float v) { return v >= 0x1p-60f && v <= 0x1p60f; }

// Replica cap of TP index j: M_j = floor(G / tau_j) = G >> j (tau_j = 2^j),
// computed rather than read from a parameter array: a kernel-parameter read
// at a runtime index is a constant-cache load (measured 300-700 cycles), a
// shift is one instruction.
__device__ __forceinline__ int rep_cap(const Dims& d, int j) { return d.G >> j; }
__device__ __forceinline__ float rep_capf(const Dims& d, int j) { return (float)(d.G >> j); }

// Fulfilment of n replicas of capacity c: min(1, (n c) / lambda), Section 3
// (Eqs. 2 and 4, r_i = x_i / lambda_i): one IEEE rounding for the product, one
// for the quotient, then the cap at 1.
__device__ __forceinline__ float fulfil(float n, float c, float lam) {
  float r = __fdiv_rn(__fmul_rn(n, c), lam);
  return fminf(r, 1.0f);
}

// The same value, the quotient by Markstein's method; rlam = RN(1/lam).
// Requires n c in {0} or [2^-60, 2^60] and lam in [2^-60, 2^60].
__device__ __forceinline__ float fulfil_fast(float n, float c, float lam, float rlam) {
  return fminf(div_markstein(__fmul_rn(n, c), lam, rlam), 1.0f);
}

// The same value for any inputs: Markstein when the product and lambda are
// in range, else the IEEE divide.
__device__ __forceinline__ float fulfil_r(float n, float c, float lam, float rlam) {
  const float x = __fmul_rn(n, c);
  if ((x == 0.0f || in_markstein_range(x)) && in_markstein_range(lam))
    return fminf(div_markstein(x, lam, rlam), 1.0f);
  return fminf(__fdiv_rn(x, lam), 1.0f);
}

// Every n c with 1 <= n <= 32767 stays in {0} or [2^-60, 2^60].
__device__ __forceinline__ bool row_in_range(float c, float lam) {
  return (c == 0.0f || (c >= 0x1p-60f && c <= 0x1p44f)) && in_markstein_range(lam);
}

// Smallest n in [1, M] with fulfil(n, c) >= t, or 0 if none (fulfil is
// nondecreasing in n under round-to-nearest). The real-valued answer is
// t lambda / c; the rounded fulfilment differs from n c / lambda by at most
// two roundings (relative 2^-22), so for n <= 32767 the answer is within one
// of ceil(t lambda / c) even with an approximate division. Five candidates
// around that estimate are tested at once; a plain bisection is kept for the
// case the bracket does not hold.
// Replica counts are handled as floats (integers up to 32767 are exact there),
// so that no integer/float conversion sits on the dependent chain; M is the
// replica cap as a float.
template <bool FAST>
__device__ __forceinline__ int min_replicas_impl(float t, float c, float lam, float rlam, float M) {
  auto f = [&](float n) { return FAST ? fulfil_fast(n, c, lam, rlam) : fulfil(n, c, lam); };
  const float fM = f(M);
  const float y = ceilf(__fdividef(__fmul_rn(t, lam), c));  // estimate only
  if (!(fM >= t)) return 0;  // also covers c == 0
  const float n = fminf(fmaxf(y, 1.0f), M);
  const float a = fmaxf(1.0f, n - 2.0f), b = fminf(M, n + 2.0f);
  const bool left = a == 1.0f || f(a - 1.0f) < t;
  const bool right = f(b) >= t;
  if (left && right) {
    float r = b;
#pragma unroll
    for (int k = 3; k >= 0; --k) {
      const float v = a + (float)k;
      if (v < b && f(v) >= t) r = v;
    }
    return (int)r;
  }
  int lo = 1, hi = (int)M;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (f((float)mid) >= t) hi = mid; else lo = mid + 1;
  }
  return lo;
}

__device__ __forceinline__ int min_replicas(float t, float c, float lam, float rlam, float M) {
  if (!(M >= 1.0f)) return 0;
  return row_in_range(c, lam) ? min_replicas_impl<true>(t, c, lam, rlam, M)
                              : min_replicas_impl<false>(t, c, lam, rlam, M);
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of the 4x32
// S-box (two 32x32->64 products) with the Weyl key schedule.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)0xD2511F53u * c.x;  // one wide multiply gives both halves
    const uint64_t p1 = (uint64_t)0xCD9E8D57u * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ k0, (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ k1, (uint32_t)p0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

// The ten round keys of one key, computed once and reused for many counters.
struct PhiloxKeys {
  uint32_t k0[10], k1[10];
};

__device__ __forceinline__ PhiloxKeys philox_keys(uint32_t k0, uint32_t k1) {
  PhiloxKeys k;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    k.k0[r] = k0 + (uint32_t)r * 0x9E3779B9u;
    k.k1[r] = k1 + (uint32_t)r * 0xBB67AE85u;
  }
  return k;
}

// The same rounds with the round keys of problem 0 from the plan.
__device__ __forceinline__ uint4 philox4x32_10_plan(uint4 c, const Plan& pl) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)0xD2511F53u * c.x;
    const uint64_t p1 = (uint64_t)0xCD9E8D57u * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ pl.rk0[r], (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ pl.rk1[r],
                   (uint32_t)p0);
  }
  return c;
}

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, const PhiloxKeys& k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)0xD2511F53u * c.x;
    const uint64_t p1 = (uint64_t)0xCD9E8D57u * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ k.k0[r], (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ k.k1[r],
                   (uint32_t)p0);
  }
  return c;
}

// lo + (hi - lo) q rounded step by step, clamped into [lo, hi]; d = hi - lo.
__device__ __forceinline__ float map_into(float lo, float d, float hi, float q) {
  float v = __fadd_rn(lo, __fmul_rn(d, q));
  return fminf(fmaxf(v, lo), hi);
}

// rint(g * 2^40) for 0 <= g <= 1, round half to even, with integer and fp32
// ALU operations only (a float-to-int64 conversion would use the FP64 unit).
// Below 2^23, adding 2^23 rounds to an integer whose value is the bit
// pattern's offset from that of 2^23; from 2^23 up the product is already
// an integer: its 24-bit significand shifted by (exponent - 23).
__device__ __forceinline__ uint64_t fixed40(float g) {
  const float x = __fmul_rn(g, 0x1p40f);
  const uint32_t small = __float_as_uint(__fadd_rn(x, 0x1p23f)) - 0x4B000000u;
  const uint32_t b = __float_as_uint(x);
  const uint32_t sh = (b >> 23) - 150u;
  const uint64_t big = (uint64_t)((b & 0x7FFFFFu) | 0x800000u) << (sh & 63u);
  return x < 0x1p23f ? (uint64_t)small : big;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch: wait for the preceding kernel of the stream
// (its writes visible), and let the next one start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------- TMA bulk copy

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Global -> shared bulk copy (no tensor map, no multicast); dst, src and
// bytes must be multiples of 16. Completion is counted on bar.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Bounded wait for phase `parity` of bar: true when it completed, false when
// limit_ns elapsed (or an iteration cap was hit) first.
__device__ __forceinline__ bool mbar_try(uint32_t a, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(a), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  const uint32_t a = smem_u32(bar);
  if (mbar_try(a, parity)) return true;  // the common case: no clock read
  const uint64_t t0 = global_ns();
  for (uint32_t it = 0; it < (1u << 28); ++it) {
    if (mbar_try(a, parity)) return true;
    if ((it & 15u) == 15u && global_ns() - t0 > limit_ns) return false;
  }
  return false;
}

// Plain arrival (no transaction bytes) on bar.
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s

// ---------------------------------------------------------------- launchers (host)

void note_launch();
// Raises the dynamic shared memory limit of kernel `func` to at least `bytes`.
// The limit belongs to the function, not to a model: models of every size and
// the allocation-free path share it, and a caller that has set it once skips
// the call later (LaunchCache), so it is only ever raised, to the largest size
// asked for so far.
cudaError_t raise_smem_limit(const void* func, size_t bytes);
// Launch with programmatic stream serialisation: the kernel may start while
// its predecessor drains and synchronises with it through pdl_wait().
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  note_launch();
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Per-model launch state: whether floors are set, and the launch shapes
// (filled on first use) per kernel instance: [floors] for the solve and the
// preparation, [path][floors] for the scorer (plain, dump, table over one
// problem, table over several).
// The preparation's and the scorer's instances are indexed by mode = floors +
// 2 prior (0..3).
constexpr int kScoreVariants = 4;
struct LaunchCache {
  int floors = 0;  // some class has a floor > 0: launch the kernel instances with floors
  size_t solve_smem[2] = {0, 0}, prep_smem[4] = {0, 0, 0, 0};
  size_t score_smem[kScoreVariants][4] = {};
  // resident blocks per SM of 256, 128 and 64 threads
  int score_blocks_per_sm[kScoreVariants][4][3] = {};
};

cudaError_t launch_qtable(float* qn, int Q, cudaStream_t s);
// Base or explicit realisations: realisation r of `n` reads cap/tail either
// from the problem set's bounds (explicit == nullptr: r = 2 p + sigma) or from
// cap_x / tail_x [n][cells].
// tstar_only: the allocations' per-class choice is not needed (the scoring
// call reads only t* and the thresholds); total_gpus is then -1 unless the
// model has floors.
cudaError_t launch_solve(const Set& set, int n, const float* cap_x, const float* tail_x,
                         fs_allocation* out, bool write_theta, LaunchCache& lc, cudaStream_t s,
                         bool tstar_only = false);
// early: the candidate ids and bounds were complete before the preceding
// kernel started, so the bounds-only work may run before the PDL wait.
// Blocks of 256 threads, or of 64 when the launch holds more than two waves
// of 256-thread blocks (sm_count SMs): each block is mostly a chain of
// dependent latencies, so more of them in flight per SM finish sooner.
// th_cap > 0: a bound on both base solves' threshold counts small enough that
// the solves build row tables (4K th_cap <= kRowTabMax); shared memory then
// holds th_cap thresholds instead of theta_cap, so that more blocks fit an SM
// (a count above it is reported as ST_TABLE, never read past).
cudaError_t launch_prep(const Set& set, const Items& it, const Plan& pl, float* tables,
                        uint64_t* sums, bool early, int sm_count, LaunchCache& lc, cudaStream_t s,
                        int th_cap = 0);
cudaError_t launch_score(const Set& set, const Items& it, const Plan& pl, const float* tables,
                         uint64_t* sums, void* dump, int dump_stride, int sm_count, LaunchCache& lc,
                         cudaStream_t s);
// status_copy (nullable): the status word as it stands after the whole call.
// part: 2 finalize_blocks(it) words of scratch (nullable when that is 0).
constexpr int kFinalizeMaxBlocks = 64;
int finalize_blocks(const Items& it);
cudaError_t launch_finalize(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                            double* gap, double* score, float* gamma_t, int32_t* best, uint32_t* status_copy,
                            uint64_t* part, cudaStream_t s);
cudaError_t launch_watchdog(uint32_t* status, uint64_t limit_ns, cudaStream_t s);
// Measurement only: median time of `reps` launches of the table path's draws
// alone (mode 0) or with its per-sample lookup (mode 1), W = 2^w, at least
// `calls` Philox calls over one wave of 128-thread blocks (synchronous).
cudaError_t draw_floor(int mode, int w, long long calls, int reps, int sm_count, double* ms_median,
                       long long* calls_done);

// tiers 3-4 and the goodput stage (fs_lex.cu)
constexpr size_t kLexCellBytes = 16;  // one cell of the programme over classes and GPUs
size_t lex_scratch_cells(const Dims& d);  // (K + 1)(G + 1) cells per realisation
// Realisations [0, n) (as launch_solve reads them; their tier-2 allocations in
// out / the base), per_launch of them at a time through scratch.
cudaError_t launch_solve_lex(const Set& set, int n, const float* cap_x, const float* tail_x, fs_allocation* out,
                             void* scratch, int per_launch, cudaStream_t s);
// Threads per block of the goodput scorer (a multiple of 32, at most 256) and
// its dynamic shared memory, or 0 when one warp's share does not fit.
constexpr size_t kGoodputSmemMax = 220 * 1024;  // of the 227 KB a block may opt into, less its static arrays
int goodput_threads(const Dims& d, const Plan& pl, bool rf, size_t* smem);
cudaError_t launch_score_goodput(const Set& set, const Items& it, const Plan& pl, const float* tables,
                                 uint64_t* sums, int floors, int sm_count, cudaStream_t s);
cudaError_t launch_finalize_goodput(const Set& set, const Items& it, const Plan& pl, const uint64_t* sums,
                                    double lam_sum, double* gap, double* score, double* gamma, int32_t* best,
                                    uint32_t* status_copy, cudaStream_t s);

// replay
struct ReplayState {
  const float* truth;     // [P][2][cells] cap, tail
  const int* perm;        // [P][cells]
  int* rounds;            // [P]
  int* state;             // [P]  -1 running, 0 undecided stop, 1 certified feasible, 2 certified infeasible
  double* gpu_seconds;    // [P]
  int* reveal_order;      // [P][cells]
  int* n_revealed;        // [P]
  float* gamma_trace;     // [P][max_rounds + 1]
  fs_allocation* final_minus;  // [P]
  int* active;            // [P] compact list of running problems
  int* n_active;          // [1]
  int* item_p;            // [P * cells]
  int* item_cell;         // [P * cells]
  int max_rounds;
  float eps;
};
// prior: DEVICE [4][cells] bounds every stream starts from.
cudaError_t launch_replay_init(const Set& set, const ReplayState& rs, const float* prior, int r0,
                               cudaStream_t s);
// Certificate of every running stream; with per > 0 also each running
// stream's list of per candidates (items [slot][per]).
cudaError_t launch_replay_certify(const Set& set, const ReplayState& rs, int round, int per, cudaStream_t s);
cudaError_t launch_replay_next(const Set& set, const ReplayState& rs, int n_active, cudaStream_t s);
cudaError_t launch_replay_reveal(const Set& set, const ReplayState& rs, const Items& it,
                                 const Plan& pl, const uint64_t* sums, int n_active, cudaStream_t s);

}  // namespace fs
