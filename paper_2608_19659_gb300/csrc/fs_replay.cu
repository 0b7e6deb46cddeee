// Profiling loop (Algorithm 1) batched over many reveal orders, for sm_103a.
//
// Every stream k is one problem of the set: its own bounds, revealed flags
// and hidden truth. A round runs, for all streams still going:
//   A-, A+ (k_solve) -> certificate (Section 4.2) and candidate list (the
//   unrevealed cells in the stream's reveal order; one kernel) -> k_prep / k_score
//   (Section 4.3) -> argmax -> reveal (interval collapses to the truth; under
//   the monotone prior the rest of its row is refit, Section 4.1).
// The fixed-order policy skips the scoring and reveals the next cell of the
// stream's order.
// The host only reads the number of streams still going once per round.
#include <cuda_runtime.h>

#include "fs_internal.cuh"
#include "fs_finalize.cuh"

namespace fs {

__device__ __forceinline__ void reveal_cell(const Set& set, const ReplayState& rs, int p, int c) {
  const Dims& d = set.d;
  float* bp = set.bounds + (size_t)p * 4 * d.cells;
  const float tc = rs.truth[((size_t)p * 2) * d.cells + c];
  const float tl = rs.truth[((size_t)p * 2 + 1) * d.cells + c];
  refit_cell(bp, d.cells, d.B, set.prior, c, tc, tl);  // collapse c; under the prior, refit its row
  set.revealed[(size_t)p * d.cells + c] = 1;
  const int q = rs.n_revealed[p]++;
  rs.reveal_order[(size_t)p * d.cells + q] = c;
  rs.gpu_seconds[p] += 300.0 * (double)(1 << ((c / d.B) & 3));  // 300 s per cell x TP GPUs
}

// One block per stream: its bounds from the common prior, an empty reveal
// order, then (thread 0) the initial design's reveals.
__global__ void k_replay_init(Set set, ReplayState rs, const float* prior, int r0) {
  const int p = blockIdx.x;
  const int cells = set.d.cells;
  float* bp = set.bounds + (size_t)p * 4 * cells;
  for (int q = threadIdx.x; q < 4 * cells; q += blockDim.x) bp[q] = prior[q];
  for (int q = threadIdx.x; q < cells; q += blockDim.x) rs.reveal_order[(size_t)p * cells + q] = -1;
  __syncthreads();
  if (threadIdx.x != 0) return;
  rs.n_revealed[p] = 0;
  rs.gpu_seconds[p] = 0.0;
  rs.rounds[p] = 0;
  rs.state[p] = -1;
  for (int q = 0; q < r0; ++q) reveal_cell(set, rs, p, rs.perm[(size_t)p * cells + q]);
}

// Certificate of every running stream, one warp per stream; collects the ones
// that go on, and (per > 0) writes each one's candidate list: its unrevealed
// cells in reveal order, 32 cells of the order at a time, each lane's place in
// the list from a ballot of the unrevealed ones before it.
__global__ void k_replay_certify(Set set, ReplayState rs, int round, int per) {
  const int p = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (p >= set.P || rs.state[p] >= 0) return;  // (the warp's lanes agree)
  const Dims& d = set.d;
  const fs_allocation& am = set.base[2 * p];
  const fs_allocation& ap = set.base[2 * p + 1];
  const float gt = __fsub_rn(ap.t_star, am.t_star);
  if (lane == 0) rs.gamma_trace[(size_t)p * (rs.max_rounds + 1) + round] = gt;
  bool known = true;  // every cell A- commits replicas to is revealed
  for (int i = lane; i < d.K; i += 32) {
    if (am.replicas[i] <= 0) continue;
    const int j = __ffs(am.tp[i]) - 1;
    const int c = (i * 4 + j) * d.B + am.bin[i];
    if (!set.revealed[(size_t)p * d.cells + c]) known = false;
  }
  known = __all_sync(0xffffffffu, known);
  // Section 4.2: infeasible when even A+ misses a critical floor; feasible
  // when A- meets the floors, the gap is within eps and A-'s cells are known
  int st = -1;
  if (!ap.floors_met) st = 2;
  else if (am.floors_met && gt <= rs.eps && known) st = 1;
  else if (round >= rs.max_rounds || rs.n_revealed[p] >= d.cells) st = 0;
  if (st >= 0) {
    if (lane == 0) {
      rs.state[p] = st;
      rs.rounds[p] = round;
    }
    const uint32_t* src = reinterpret_cast<const uint32_t*>(&am);
    uint32_t* dst = reinterpret_cast<uint32_t*>(rs.final_minus + p);
    for (int w = lane; w < (int)(sizeof(fs_allocation) / 4); w += 32) dst[w] = src[w];
    return;
  }
  int a = 0;
  if (lane == 0) {
    a = atomicAdd(rs.n_active, 1);
    rs.active[a] = p;
  }
  a = __shfl_sync(0xffffffffu, a, 0);
  if (per <= 0) return;
  int q = 0;
  for (int k0 = 0; k0 < d.cells && q < per; k0 += 32) {
    const int k = k0 + lane;
    const int c = k < d.cells ? rs.perm[(size_t)p * d.cells + k] : 0;
    const bool open = k < d.cells && !set.revealed[(size_t)p * d.cells + c];
    const uint32_t bal = __ballot_sync(0xffffffffu, open);
    const int at = q + __popc(bal & ((1u << lane) - 1u));
    if (open && at < per) {
      rs.item_p[(size_t)a * per + at] = p;
      rs.item_cell[(size_t)a * per + at] = c;
    }
    q += __popc(bal);
  }
  if (lane == 0 && q < per) atomicOr(set.status, ST_TABLE);
}

// Fixed-order policy: running stream slot a reveals its next unrevealed cell
// in reveal order (the candidate list's first entry).
__global__ void k_replay_next(Set set, ReplayState rs, int n_active) {
  const int a = blockIdx.x * blockDim.x + threadIdx.x;
  if (a >= n_active) return;
  const int p = rs.active[a];
  const Dims& d = set.d;
  for (int k = 0; k < d.cells; ++k) {
    const int c = rs.perm[(size_t)p * d.cells + k];
    if (!set.revealed[(size_t)p * d.cells + c]) {
      reveal_cell(set, rs, p, c);
      return;
    }
  }
  atomicOr(set.status, ST_TABLE);  // a running stream always has an unrevealed cell
}

__global__ void k_replay_reveal(Set set, ReplayState rs, Items it, Plan pl, const uint64_t* sums, int per) {
  const int a = blockIdx.x;
  const int p = rs.active[a];
  const Best b = finalize_problem(set, it, pl, sums, p, a * per, (a + 1) * per, nullptr, nullptr, nullptr, a * per);
  if (threadIdx.x == 0 && b.valid()) reveal_cell(set, rs, p, b.cell);
}

cudaError_t launch_replay_init(const Set& set, const ReplayState& rs, const float* prior, int r0,
                               cudaStream_t s) {
  note_launch();
  k_replay_init<<<set.P, 128, 0, s>>>(set, rs, prior, r0);
  return cudaGetLastError();
}

cudaError_t launch_replay_certify(const Set& set, const ReplayState& rs, int round, int per, cudaStream_t s) {
  note_launch();
  k_replay_certify<<<(set.P + 3) / 4, 128, 0, s>>>(set, rs, round, per);
  return cudaGetLastError();
}

cudaError_t launch_replay_next(const Set& set, const ReplayState& rs, int n_active, cudaStream_t s) {
  note_launch();
  k_replay_next<<<(n_active + 127) / 128, 128, 0, s>>>(set, rs, n_active);
  return cudaGetLastError();
}

cudaError_t launch_replay_reveal(const Set& set, const ReplayState& rs, const Items& it, const Plan& pl,
                                 const uint64_t* sums, int n_active, cudaStream_t s) {
  note_launch();
  k_replay_reveal<<<n_active, 256, 0, s>>>(set, rs, it, pl, sums, it.n / n_active);
  return cudaGetLastError();
}

}  // namespace fs
