// Scoring without any device allocation.
//
// Some callers cannot allocate device memory while they run: processes whose
// device memory is already handed out by their own pool (a cudaMalloc would
// fail or fragment it), and latency-critical paths that must not pay for
// cudaMalloc / cudaFree, which can synchronise the whole device.
// fs_score_candidates_noalloc serves them: the caller passes the inputs and the
// outputs in device memory, and every intermediate (base solves, threshold
// lists, per-candidate tables, fixed-point sums, status word) lives in one
// file-scope device array of fixed size, kStaticScratchBytes. That array exists
// on every GPU that loads this library, for as long as the process lives.
//
// Host code cannot use the array's name as a device address, so the first call
// on each device looks the address up with cudaGetSymbolAddress (with that
// device current) and keeps it; that first call should therefore come before
// any stream capture. All calls share the array and it keeps whatever the last
// call left in it: the status word is cleared by every call, and the kernels
// overwrite or clear everything else before reading it. Calls whose GPU work
// overlaps (two streams, two host threads) race on the array.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "fs_internal.cuh"

namespace fs {

int record_error(int code, const char* msg);

constexpr size_t kStaticScratchBytes = 16u << 20;  // 16 MiB per device
constexpr int kMaxStaticDevices = 64;

}  // namespace fs

static __device__ __align__(256) unsigned char g_fs_static_scratch[fs::kStaticScratchBytes];

namespace {

using namespace fs;

std::mutex g_static_mu;
void* g_static_ptr[kMaxStaticDevices] = {};
LaunchCache g_static_lc[kMaxStaticDevices];

int say(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  return record_error(code, buf);
}

int cuda_say(cudaError_t e, const char* what) {
  return say(FS_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t up256(size_t x) { return (x + 255) / 256 * 256; }

bool pow2(long long x) { return x > 0 && (x & (x - 1)) == 0; }

}  // namespace

extern "C" int fs_score_candidates_noalloc(int32_t K, int32_t B, int32_t G, const float* bounds_dev,
                                           const float* slo_dev, const float* demand_dev,
                                           const float* quantile_dev, int32_t Q, const fs_samples* smp,
                                           double* gap_dev, double* score_dev, float* gamma_t_dev,
                                           int32_t* best_dev, void* cuda_stream) {
  // --- sizes (device data cannot be inspected here; see the header)
  if (K < 1 || K > FS_MAX_CLASSES) return say(FS_EINVAL, "K = %d outside [1, %d]", K, FS_MAX_CLASSES);
  if (B < 1 || B > FS_MAX_BINS) return say(FS_EINVAL, "B = %d outside [1, %d]", B, FS_MAX_BINS);
  if (G < 1 || G > FS_MAX_GPUS) return say(FS_EINVAL, "G = %d outside [1, %d]", G, FS_MAX_GPUS);
  if (!bounds_dev || !slo_dev || !demand_dev) return say(FS_EINVAL, "bounds / slo / demand is NULL");
  const long long theta_cap = (long long)K * ((G >> 0) + (G >> 1) + (G >> 2) + (G >> 3));
  if (theta_cap > FS_MAX_THRESHOLDS)
    return say(FS_EINVAL, "K * sum floor(G/tau) = %lld exceeds %d", theta_cap, FS_MAX_THRESHOLDS);
  if (quantile_dev) {
    if (!pow2(Q) || Q < 4 || Q > (1 << 24)) return say(FS_EINVAL, "Q = %d must be a power of two in [4, 2^24]", Q);
  } else {
    Q = 4096;
  }
  if (!smp) return say(FS_EINVAL, "samples is NULL");
  const int n = smp->n_cand;
  if (n < 0) return say(FS_EINVAL, "n_cand < 0");
  if (n > 0 && !smp->cand) return say(FS_EINVAL, "cand is NULL");
  if (!pow2(smp->O) || smp->O > Q) return say(FS_EINVAL, "O = %d must be a power of two <= Q = %d", smp->O, Q);
  if (Q / smp->O > 16384) return say(FS_EINVAL, "Q / O exceeds 16384 quantiles per stratum");
  if (smp->S < 1) return say(FS_EINVAL, "S = %d < 1", smp->S);
  if ((long long)smp->O * smp->S > FS_MAX_SAMPLES_PER_CAND) return say(FS_EINVAL, "O * S exceeds 2^22");

  Dims d{};
  d.K = K;
  d.B = B;
  d.G = G;
  d.Q = Q;
  d.cells = K * 4 * B;
  d.K4 = 4 * K;
  d.theta_cap = (int)theta_cap;
  d.lcap = 4;
  while (d.lcap < d.theta_cap + 1) d.lcap <<= 1;
  d.slot_floats = kTableHeader + 3 * d.lcap;

  // --- layout of the static scratch for this call
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = up256(off + bytes);
    return o;
  };
  const size_t o_status = take(4), o_work = take(32), o_part = take(16 * (size_t)kFinalizeMaxBlocks);
  const size_t o_qn = quantile_dev ? 0 : take(4 * (size_t)Q);
  const size_t o_theta = take(8 * (size_t)d.theta_cap), o_nth = take(8);
  const size_t o_rowc = take(8 * (size_t)d.K4), o_rowb = take(8 * (size_t)d.K4);
  const size_t o_base = take(2 * sizeof(fs_allocation));
  const size_t o_rtab = take(8 * (size_t)kRowTabMax);  // row tables of the two base solves
  const int Wq = Q / smp->O, Wp = 4 + ((Wq + 3) & ~3);
  const size_t item_floats = 2 * (size_t)d.slot_floats + (size_t)smp->O * Wp;
  const size_t o_tab = take((size_t)std::max(n, 1) * item_floats * 4);
  const size_t o_sums = take((size_t)std::max(n, 1) * smp->O * 8);
  if (off > kStaticScratchBytes)
    return say(FS_EINVAL,
               "this call needs %zu bytes of scratch; the allocation-free entry point has %zu "
               "(score fewer candidates per call, or use fs_score_candidates)",
               off, kStaticScratchBytes);

  // --- per-device set-up: the array's device address, looked up once
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_say(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxStaticDevices) return say(FS_EINVAL, "device %d beyond %d", dev, kMaxStaticDevices);
  char* base = nullptr;
  LaunchCache lc;  // this call's copy of the device's launch shapes, written back under the lock
  {
    std::lock_guard<std::mutex> lock(g_static_mu);
    if (!g_static_ptr[dev]) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_fs_static_scratch);
      if (e != cudaSuccess) return cuda_say(e, "cudaGetSymbolAddress(static scratch)");
      g_static_ptr[dev] = p;
    }
    base = static_cast<char*>(g_static_ptr[dev]);
    lc = g_static_lc[dev];
  }
  int sm_count = 0;
  e = cudaDeviceGetAttribute(&sm_count, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_say(e, "device query");

  Set set{};
  set.d = d;
  set.P = 1;
  set.lam = demand_dev;
  set.slo = slo_dev;
  set.qn = quantile_dev ? quantile_dev : reinterpret_cast<const float*>(base + o_qn);
  set.bounds = const_cast<float*>(bounds_dev);  // the scoring kernels only read the bounds
  set.revealed = nullptr;
  set.theta = reinterpret_cast<float*>(base + o_theta);
  set.ntheta = reinterpret_cast<int*>(base + o_nth);
  set.rowC = reinterpret_cast<float*>(base + o_rowc);
  set.rowB = reinterpret_cast<int*>(base + o_rowb);
  set.base = reinterpret_cast<fs_allocation*>(base + o_base);
  set.status = reinterpret_cast<uint32_t*>(base + o_status);
  set.work = reinterpret_cast<unsigned long long*>(base + o_work);
  set.skip = nullptr;
  set.rtab = reinterpret_cast<int*>(base + o_rtab);
  set.prior = 0;  // the revealed-only prior: no cell is measured here

  Items it{};
  it.n = n;
  it.p = nullptr;
  it.cell = smp->cand;
  it.off = nullptr;
  Plan pl{};
  pl.key0 = (uint32_t)smp->seed;
  pl.key1 = (uint32_t)(smp->seed >> 32);
  pl.stream_base = smp->stream_id;
  pl.round = smp->round;
  pl.O = smp->O;
  pl.S = smp->S;
  pl.W = Q / smp->O;
  pl.w = 0;
  while ((1 << pl.w) < pl.W) ++pl.w;
  pl.sh = 16 - pl.w;
  pl.logO = 0;
  while ((1 << pl.logO) < pl.O) ++pl.logO;
  pl.calls = (smp->S + 3) / 4;
  pl.Wp = Wp;
  pl.item_floats = (long long)item_floats;
  plan_round_keys(pl);

  // --- the scoring pipeline on the caller's stream, then wait and report
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  e = cudaMemsetAsync(set.status, 0, 4, s);  // the array keeps the last call's status word
  if (e == cudaSuccess && !quantile_dev) e = launch_qtable(const_cast<float*>(set.qn), Q, s);
  if (e == cudaSuccess) e = launch_solve(set, 2, nullptr, nullptr, nullptr, true, lc, s, true);
  if (e == cudaSuccess) e = launch_prep(set, it, pl, reinterpret_cast<float*>(base + o_tab),
                                        reinterpret_cast<uint64_t*>(base + o_sums), true, sm_count, lc, s);
  if (e == cudaSuccess)
    e = launch_score(set, it, pl, reinterpret_cast<const float*>(base + o_tab),
                     reinterpret_cast<uint64_t*>(base + o_sums), nullptr, 0, sm_count, lc, s);
  if (e == cudaSuccess)
    e = launch_finalize(set, it, pl, reinterpret_cast<const uint64_t*>(base + o_sums), gap_dev, score_dev,
                        gamma_t_dev, best_dev, nullptr, reinterpret_cast<uint64_t*>(base + o_part), s);
  {
    // launch shapes only grow (a kernel's shared-memory limit is only raised):
    // keep the larger of what this call and any concurrent one found
    std::lock_guard<std::mutex> lock(g_static_mu);
    LaunchCache& g = g_static_lc[dev];
    for (int f = 0; f < 2; ++f) g.solve_smem[f] = std::max(g.solve_smem[f], lc.solve_smem[f]);
    for (int f = 0; f < 4; ++f) {
      g.prep_smem[f] = std::max(g.prep_smem[f], lc.prep_smem[f]);
      for (int v = 0; v < kScoreVariants; ++v)
        if (lc.score_smem[v][f] && lc.score_smem[v][f] != g.score_smem[v][f]) {
          g.score_smem[v][f] = lc.score_smem[v][f];
          g.score_blocks_per_sm[v][f][0] = lc.score_blocks_per_sm[v][f][0];
          g.score_blocks_per_sm[v][f][1] = lc.score_blocks_per_sm[v][f][1];
          g.score_blocks_per_sm[v][f][2] = lc.score_blocks_per_sm[v][f][2];
        }
    }
  }
  if (e != cudaSuccess) return cuda_say(e, "launch (allocation-free scoring)");
  uint32_t st = 0;
  e = cudaMemcpyAsync(&st, set.status, 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_say(e, "synchronize (allocation-free scoring)");
  if (st & ST_TIMEOUT) return say(FS_ETIMEOUT, "a device wait timed out (status 0x%x)", st);
  if (st) return say(FS_EDEVICE, "device status word 0x%x", st);
  return FS_OK;
}
