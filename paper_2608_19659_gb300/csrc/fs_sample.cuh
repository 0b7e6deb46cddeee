// Table-path sampling and the row capacity of a scenario, shared by the
// Monte-Carlo kernels of the max-min stage (fs_score.cu) and the goodput
// stage (fs_lex.cu).
#pragma once

#include "fs_internal.cuh"

namespace fs {

// Row r's capacity in a scenario under the monotone prior (see k_prep):
// max(g ? max(P_open, c_y) : P_closed, min(max(c_y, F_lo), F_hi)).
struct RowCap {
  float pc, po, lf, hf;
};

__device__ __forceinline__ RowCap row_cap_of(const float* h) { return RowCap{h[H_CX], h[H_PO], h[H_LF], h[H_HF]}; }

__device__ __forceinline__ float row_cap(const RowCap& r, float cy, bool g) {
  return fmaxf(g ? fmaxf(r.po, cy) : r.pc, fminf(fmaxf(cy, r.lf), r.hf));
}

// Philox calls [q_lo, q_hi) of one segment on the table path: the sum of the
// drawn entries (each rint(gap 2^40) <= 2^40, stored as one 64-bit word).
// Per sample: the capacity position floor(word W / 2^32), the word's top w
// bits for W = 2^w; the tail gate, (word & 0xFFFF) < kgs, as
// (word * 65536 mod 2^32) < kgs16 with kgs16 = min(kgs 2^16, 2^32 - 1) (a
// multiply-add and a compare); the entry's shared address base + index * 8 (a
// multiply-add); its load and one 64-bit add. Two calls per iteration give two
// independent Philox chains. KC: one problem, its round keys read from the
// plan. GATE = false: the stratum's tail gate is the same at every position
// (its mapped tails all pass the SLO, or none does; known from the
// preparation's gate position), so the entry is the capacity position's in
// the table at gtab_s with a stride of `stride` bytes (the open half, or under
// the prior the closed half; without the prior a closed stratum's entries are
// all the closed-gate value, stored once: stride 0, so a warp's loads are one
// broadcast) and no scenario tests the gate.
template <bool KC>
__device__ __forceinline__ uint4 draw_call(const Plan& pl, const PhiloxKeys& keys, uint32_t q, uint32_t ctr1,
                                           uint32_t ctr2, uint32_t ctr3) {
  if constexpr (KC) return philox4x32_10_plan(make_uint4(q, ctr1, ctr2, ctr3), pl);
  else return philox4x32_10(make_uint4(q, ctr1, ctr2, ctr3), keys);
}

template <bool KC, bool RF, bool GATE = true>
__device__ __forceinline__ uint64_t sample_gtab(const Plan& pl, const PhiloxKeys& keys, int o, int cell, int q_lo,
                                                int q_hi, uint32_t gtab_s, uint32_t kgs16, uint32_t stride = 8u) {
  const uint32_t ctr1 = (uint32_t)o, ctr2 = (uint32_t)cell, ctr3 = pl.round;
  const uint32_t W = (uint32_t)pl.W, w = (uint32_t)pl.w;
  const uint32_t mul = pl.lo16_mul, eb = GATE ? pl.entry_bytes : stride;
  uint64_t total = 0;
  auto take = [&](uint32_t word) {
    // capacity position floor(word W / 2^32): W = 2^w, so the word's top w
    // bits, taken by a funnel shift (0 for w = 0) on the shift unit rather
    // than the integer multiplier, which the Philox rounds keep busy
    const uint32_t cap = __funnelshift_lc(word, 0u, w);
    const uint32_t idx = !GATE ? cap : word * mul < kgs16 ? cap : (RF ? cap + W : W);
    uint64_t a;
    asm volatile("ld.shared.u64 %0, [%1];" : "=l"(a) : "r"(gtab_s + idx * eb));
    total += a;
  };
  auto take4 = [&](const uint4& x) {
    take(x.x);
    take(x.y);
    take(x.z);
    take(x.w);
  };
  const int q_full = min(q_hi, pl.S >> 2);  // calls whose four samples all exist
  const int step = (int)blockDim.x;
  int q = q_lo + (int)threadIdx.x;
  for (; q + step < q_full; q += 2 * step) {
    const uint4 x0 = draw_call<KC>(pl, keys, (uint32_t)q, ctr1, ctr2, ctr3);
    const uint4 x1 = draw_call<KC>(pl, keys, (uint32_t)(q + step), ctr1, ctr2, ctr3);
    take4(x0);
    take4(x1);
  }
  if (q < q_full) {
    take4(draw_call<KC>(pl, keys, (uint32_t)q, ctr1, ctr2, ctr3));
    q += step;
  }
  if (q < q_hi) {  // the segment's last call, serving S mod 4 samples
    const uint4 x = draw_call<KC>(pl, keys, (uint32_t)q, ctr1, ctr2, ctr3);
    const int nv = pl.S - 4 * q;
    take(x.x);
    if (nv > 1) take(x.y);
    if (nv > 2) take(x.z);
  }
  return total;
}

}  // namespace fs
