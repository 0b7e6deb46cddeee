// C ABI of the decision-gap scorer: model lifetime, argument checks, device
// buffers and the launch sequence of each call. See include/fleetsieve.h for
// the contract of every entry point.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "fs_internal.cuh"

namespace fs {

// An NVTX range over one call of the boundary (load, base solves, scoring,
// reveal, replay), for timeline tools; with no tool attached a push and a pop
// are two calls through a null handler.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

static std::atomic<uint64_t> g_launches{0};
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

cudaError_t raise_smem_limit(const void* func, size_t bytes) {
  static std::mutex mu;
  static std::vector<std::pair<const void*, size_t>> limits;  // (kernel, largest limit set)
  std::lock_guard<std::mutex> lock(mu);
  size_t* cur = nullptr;
  for (auto& e : limits)
    if (e.first == func) cur = &e.second;
  if (!cur) {
    limits.emplace_back(func, 0);
    cur = &limits.back().second;
  }
  const size_t want = std::max(*cur, bytes);
  const cudaError_t e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)want);
  if (e == cudaSuccess) *cur = want;
  return e;
}

static thread_local std::string g_err;

static int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

// Error message for other translation units of the library (thread-local, read
// back through fs_last_error).
int record_error(int code, const char* msg) {
  g_err = msg;
  return code;
}

static int cuda_fail(cudaError_t e, const char* what) {
  return fail(e == cudaErrorMemoryAllocation ? FS_ENOMEM : FS_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define FS_CUDA(call, what)                          \
  do {                                               \
    cudaError_t e_ = (call);                         \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

static bool is_pow2(long long x) { return x > 0 && (x & (x - 1)) == 0; }

static int log2i(long long x) {
  int v = 0;
  while ((1LL << v) < x) ++v;
  return v;
}

// One device allocation that is grown on demand (never shrunk).
struct Buf {
  void* p = nullptr;
  size_t bytes = 0;
  int ensure(size_t want, const char* what) {
    if (want <= bytes) return FS_OK;
    if (p) cudaFree(p);
    p = nullptr;
    bytes = 0;
    size_t b = std::max<size_t>(want, 256);
    cudaError_t e = cudaMalloc(&p, b);
    if (e != cudaSuccess) {
      p = nullptr;
      return cuda_fail(e, what);
    }
    bytes = b;
    return FS_OK;
  }
  void release() {
    if (p) cudaFree(p);
    p = nullptr;
    bytes = 0;
  }
};

// Page-locked host memory that grows on demand, mapped into the device's
// address space: copies to and from it are asynchronous, so a call can queue
// them and wait once, and kernels can read and write it directly (dev).
struct HostBuf {
  void* p = nullptr;
  void* dev = nullptr;
  size_t bytes = 0;
  int ensure(size_t want, const char* what) {
    if (want <= bytes) return FS_OK;
    if (p) cudaFreeHost(p);
    p = nullptr;
    dev = nullptr;
    bytes = 0;
    size_t b = std::max<size_t>(want, 256);
    cudaError_t e = cudaHostAlloc(&p, b, cudaHostAllocMapped);
    if (e == cudaSuccess) e = cudaHostGetDevicePointer(&dev, p, 0);
    if (e != cudaSuccess) {
      if (p) cudaFreeHost(p);
      p = nullptr;
      dev = nullptr;
      return cuda_fail(e, what);
    }
    bytes = b;
    return FS_OK;
  }
  void release() {
    if (p) cudaFreeHost(p);
    p = nullptr;
    dev = nullptr;
    bytes = 0;
  }
};

}  // namespace fs

using namespace fs;

struct fs_model {
  Dims d{};
  int device = 0;
  int sm_count = 0;
  cudaStream_t stream = nullptr;
  // device state of the single problem (P = 1)
  Buf fixed;      // lam, slo + floors, qn, bounds, revealed, theta, ntheta, rowC, rowB, base, status
  Set set{};
  // per-call scratch
  Buf cand, tables, sums, outs, real, lex;
  Buf replay;     // fs_replay's state of every stream (grown on demand, kept)
  int objective = FS_OBJECTIVE_MAXMIN;  // FS_OBJECTIVE_LEXICOGRAPHIC: fs_solve* and the certificate to tier 4
  // host mirrors
  std::vector<float> h_bounds;      // [4][cells]
  std::vector<uint8_t> h_revealed;  // [cells]
  std::vector<float> h_lam, h_slo, h_dlt;
  // page-locked staging: the last bounds upload (its copy may still be in
  // flight until up_done), and a synchronous call's outputs and status word
  HostBuf h_up, h_out;
  cudaEvent_t up_done = nullptr;
  bool up_pending = false;
  bool staged = false;  // the staging holds bounds the device copy does not have yet
  int th_bound = -1;    // threshold_bound of the current bounds (-1: not computed yet)
  LaunchCache lc;
  // optional timing events: 5 per timed call (before solve, prep, score,
  // finalize, and after finalize); mode 1 records only the two around score
  int timing = 0;
  std::vector<cudaEvent_t> ev;
  size_t ev_used = 0;
};

namespace {

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr size_t kMaxTimedEvents = 5 * 4096;

int check_cells(const float* a, int n, const char* name) {
  if (!a) return fail(FS_EINVAL, "%s is NULL", name);
  for (int i = 0; i < n; ++i)
    if (!std::isfinite(a[i]) || a[i] < 0.0f) return fail(FS_EINVAL, "%s[%d] = %g is not finite and >= 0", name, i, (double)a[i]);
  return FS_OK;
}

int check_bounds4(const float* clo, const float* chi, const float* tlo, const float* thi, int cells) {
  int rc;
  if ((rc = check_cells(clo, cells, "cap_lo")) || (rc = check_cells(chi, cells, "cap_hi")) ||
      (rc = check_cells(tlo, cells, "tail_lo")) || (rc = check_cells(thi, cells, "tail_hi")))
    return rc;
  for (int c = 0; c < cells; ++c) {
    if (clo[c] > chi[c]) return fail(FS_EINVAL, "cap_lo[%d] > cap_hi[%d]", c, c);
    if (tlo[c] > thi[c]) return fail(FS_EINVAL, "tail_lo[%d] > tail_hi[%d]", c, c);
  }
  return FS_OK;
}

// +0 for -0, so that nonnegative floats order like their bit patterns.
inline float canon(float v) { return v == 0.0f ? 0.0f : v; }

// The staging buffer of the last bounds upload is free once that copy has run.
int wait_upload(fs_model* m) {
  if (m->up_pending) {
    FS_CUDA(cudaEventSynchronize(m->up_done), "wait for the bounds upload");
    m->up_pending = false;
  }
  return FS_OK;
}

// Work queued on a stream other than the model's starts after the last bounds upload.
int order_after_upload(fs_model* m, cudaStream_t s) {
  if (m->up_pending && s != m->stream) FS_CUDA(cudaStreamWaitEvent(s, m->up_done, 0), "order after the upload");
  return FS_OK;
}

// Stage the host mirror's bounds and revealed flags in page-locked memory
// (once the previous staging's device copy has run). No CUDA work is queued:
// the next call that needs the bounds on the device queues the copy
// (flush_bounds), and a synchronous scoring call reads the staged bounds
// directly, so an update costs no copy-engine round trip of its own.
int stage_bounds(fs_model* m) {
  const size_t nb = m->h_bounds.size() * 4, nr = m->h_revealed.size();
  int rc = wait_upload(m);
  if (rc) return rc;
  // bounds and revealed flags lie in one span of the model's buffer (the
  // flags after the bounds' 256-byte padding): staged alike, one copy
  const size_t rev_off = (size_t)(reinterpret_cast<char*>(m->set.revealed) - reinterpret_cast<char*>(m->set.bounds));
  if ((rc = m->h_up.ensure(rev_off + nr, "bounds staging"))) return rc;
  char* h = static_cast<char*>(m->h_up.p);
  std::memcpy(h, m->h_bounds.data(), nb);
  std::memcpy(h + rev_off, m->h_revealed.data(), nr);
  m->staged = true;
  m->th_bound = -1;
  return FS_OK;
}

// An upper bound on the number of thresholds of either base solve of the
// current bounds. A row (class i, TP tau) whose best SLO-feasible capacity is
// C holds at most min(floor(G / tau), n_sat) fulfilment values, n_sat the
// first replica count whose fulfilment RN(RN(n C) / lambda_i) reaches 1: every
// n >= lambda_i / C (1 + 2^-23) does (each RN step loses at most 2^-24
// relatively), so n_sat <= floor(lambda_i / C (1 + 2^-18)) + 3, with margin for
// the bound's own double arithmetic. A row without a feasible bin holds none.
int threshold_bound(const fs_model* m) {
  const Dims& d = m->d;
  const int cells = d.cells, B = d.B;
  const float* hb = m->h_bounds.data();
  long long most = 0;
  for (int sigma = 0; sigma < 2; ++sigma) {
    const float* cap = hb + (size_t)(sigma ? CAP_HI : CAP_LO) * cells;
    const float* tail = hb + (size_t)(sigma ? TAIL_LO : TAIL_HI) * cells;
    long long tot = 0;
    for (int rho = 0; rho < d.K4; ++rho) {
      const int i = rho >> 2, M = d.G >> (rho & 3);
      bool any = false;
      float C = 0.0f;
      for (int b = 0; b < B; ++b) {
        const int c = rho * B + b;
        if (tail[c] <= m->h_slo[i]) {
          any = true;
          C = std::max(C, cap[c]);
        }
      }
      if (!any || M < 1) continue;
      long long n = M;
      if (C > 0.0f) {
        const double q = (double)m->h_lam[i] / (double)C * (1.0 + 0x1p-18);
        if (q < (double)M) n = std::min<long long>(M, (long long)q + 3);
      }
      tot += n;
    }
    most = std::max(most, tot);
  }
  return (int)std::min<long long>(most, d.theta_cap);
}

// Queue the device copy of staged bounds (if any) on the model's stream without
// waiting, and order work on stream s after the last such copy.
int flush_bounds(fs_model* m, cudaStream_t s) {
  if (m->staged) {
    const size_t span = (size_t)(reinterpret_cast<char*>(m->set.revealed) - reinterpret_cast<char*>(m->set.bounds)) +
                        m->h_revealed.size();
    FS_CUDA(cudaMemcpyAsync(m->set.bounds, m->h_up.p, span, cudaMemcpyHostToDevice, m->stream), "upload bounds");
    if (!m->up_done) FS_CUDA(cudaEventCreateWithFlags(&m->up_done, cudaEventDisableTiming), "create upload event");
    FS_CUDA(cudaEventRecord(m->up_done, m->stream), "record upload event");
    m->up_pending = true;
    m->staged = false;
  }
  return order_after_upload(m, s);
}

// Turn a nonzero device status word into an error (and clear it for the next call).
int status_error(fs_model* m, uint32_t st) {
  if (!st) return FS_OK;
  uint32_t z = 0;
  cudaMemcpy(m->set.status, &z, 4, cudaMemcpyHostToDevice);
  if (st & ST_TIMEOUT) return fail(FS_ETIMEOUT, "a device wait timed out (status 0x%x)", st);
  return fail(FS_EDEVICE, "device status word 0x%x", st);
}

// Wait for the work queued on s and check the status word: one asynchronous
// copy into page-locked memory and one synchronisation.
int read_status(fs_model* m, cudaStream_t s) {
  int rc = m->h_out.ensure(64, "status staging");
  if (rc) return rc;
  uint32_t* hs = static_cast<uint32_t*>(m->h_out.p);
  FS_CUDA(cudaMemcpyAsync(hs, m->set.status, 4, cudaMemcpyDeviceToHost, s), "read status");
  FS_CUDA(cudaStreamSynchronize(s), "synchronize");
  return status_error(m, *hs);
}

int check_samples(const fs_model* m, const fs_samples* s, bool host_cand) {
  if (!s) return fail(FS_EINVAL, "samples is NULL");
  if (s->n_cand < 0) return fail(FS_EINVAL, "n_cand < 0");
  if (s->n_cand > 0 && !s->cand) return fail(FS_EINVAL, "cand is NULL");
  if (!is_pow2(s->O) || s->O > m->d.Q) return fail(FS_EINVAL, "O = %d must be a power of two <= Q = %d", s->O, m->d.Q);
  if (m->d.Q / s->O > 16384) return fail(FS_EINVAL, "Q / O = %d exceeds 16384 quantiles per stratum", m->d.Q / s->O);
  if (s->S < 1) return fail(FS_EINVAL, "S = %d < 1", s->S);
  if ((long long)s->O * s->S > FS_MAX_SAMPLES_PER_CAND) return fail(FS_EINVAL, "O * S exceeds 2^22");
  if ((long long)s->n_cand * s->O > (1LL << 30)) return fail(FS_EINVAL, "n_cand * O too large");
  if (host_cand)
    for (int e = 0; e < s->n_cand; ++e)
      if (s->cand[e] < 0 || s->cand[e] >= m->d.cells) return fail(FS_EINVAL, "cand[%d] = %d out of range", e, s->cand[e]);
  return FS_OK;
}

Plan make_plan(const fs_model* m, const fs_samples* s, int n_items) {
  Plan pl{};
  pl.key0 = (uint32_t)s->seed;
  pl.key1 = (uint32_t)(s->seed >> 32);
  pl.stream_base = s->stream_id;
  pl.round = s->round;
  pl.O = s->O;
  pl.S = s->S;
  pl.W = m->d.Q / s->O;
  pl.w = log2i(pl.W);
  pl.sh = 16 - pl.w;
  pl.logO = log2i(s->O);
  pl.calls = (s->S + 3) / 4;
  pl.Wp = 4 + ((pl.W + 3) & ~3);
  pl.item_floats = 2LL * m->d.slot_floats + (long long)s->O * pl.Wp;
  plan_round_keys(pl);
  (void)n_items;
  return pl;
}

int ensure_items(fs_model* m, int n, int O) {
  int rc;
  if ((rc = m->cand.ensure((size_t)std::max(n, 1) * 4, "candidate list"))) return rc;
  const int W = m->d.Q / O, Wp = 4 + ((W + 3) & ~3);
  const size_t item_floats = 2 * (size_t)m->d.slot_floats + (size_t)O * Wp;
  if ((rc = m->tables.ensure((size_t)std::max(n, 1) * item_floats * 4, "candidate records"))) return rc;
  // sums, then the split reduction's scratch (2 words per block)
  if ((rc = m->sums.ensure((size_t)std::max(n, 1) * O * 8 + 16 * (size_t)kFinalizeMaxBlocks, "sums"))) return rc;
  if ((rc = m->outs.ensure((size_t)std::max(n, 1) * 16 + 64, "outputs"))) return rc;
  return FS_OK;
}

// The scoring sequence on stream s; cand_dev holds n_cand cell ids.
int run_score(fs_model* m, const Set& set, const fs_samples* smp, const int32_t* cand_dev, double* gap,
              double* score, float* gamma_t, int32_t* best, void* dump, cudaStream_t s,
              uint32_t* status_copy = nullptr) {
  const int n = smp->n_cand;
  Items it{};
  it.n = n;
  it.p = nullptr;
  it.cell = cand_dev;
  it.off = nullptr;
  const Plan pl = make_plan(m, smp, n);
  const bool timed = m->timing && n > 0 && m->ev_used + 5 <= kMaxTimedEvents;
  cudaEvent_t* ev = nullptr;
  if (timed) {
    while (m->ev.size() < m->ev_used + 5) {
      cudaEvent_t e;
      FS_CUDA(cudaEventCreate(&e), "create timing event");
      m->ev.push_back(e);
    }
    ev = &m->ev[m->ev_used];
    m->ev_used += 5;
  }
  const bool phases = timed && m->timing == 2;
  if (phases) FS_CUDA(cudaEventRecord(ev[0], s), "record timing event");
  FS_CUDA(launch_solve(set, 2, nullptr, nullptr, nullptr, true, m->lc, s, true), "launch solve");
  if (phases) FS_CUDA(cudaEventRecord(ev[1], s), "record timing event");
  if (m->th_bound < 0) m->th_bound = threshold_bound(m);
  FS_CUDA(launch_prep(set, it, pl, (float*)m->tables.p, (uint64_t*)m->sums.p, true, m->sm_count, m->lc, s,
                      m->th_bound),
          "launch prep");
  if (timed) FS_CUDA(cudaEventRecord(ev[2], s), "record timing event");
  FS_CUDA(launch_score(set, it, pl, (const float*)m->tables.p, (uint64_t*)m->sums.p, dump,
                       fs_dump_stride(m), m->sm_count, m->lc, s),
          "launch score");
  if (timed) FS_CUDA(cudaEventRecord(ev[3], s), "record timing event");
  FS_CUDA(launch_finalize(set, it, pl, (const uint64_t*)m->sums.p, gap, score, gamma_t, best, status_copy,
                          (uint64_t*)m->sums.p + (size_t)std::max(n, 1) * smp->O, s),
          "launch finalize");
  if (phases) FS_CUDA(cudaEventRecord(ev[4], s), "record timing event");
  return FS_OK;
}

// Tiers 3-4 (fs_lex.cu) of n realisations whose tier-2 allocations are in out
// (or the base), when the model's objective asks for them.
int solve_lex_pass(fs_model* m, const Set& set, int n, const float* cap_x, const float* tail_x, fs_allocation* out,
                   cudaStream_t s) {
  if (m->objective != FS_OBJECTIVE_LEXICOGRAPHIC || n <= 0) return FS_OK;
  const size_t per_real = lex_scratch_cells(m->d) * kLexCellBytes;
  const int per_launch = (int)std::max<size_t>(1, std::min<size_t>((size_t)n, (64u << 20) / per_real));
  int rc = m->lex.ensure(per_real * per_launch, "lexicographic scratch");
  if (rc) return rc;
  FS_CUDA(launch_solve_lex(set, n, cap_x, tail_x, out, m->lex.p, per_launch, s), "launch lexicographic solve");
  return FS_OK;
}

double demand_sum(const fs_model* m) {
  double t = 0.0;
  for (float v : m->h_lam) t += (double)v;
  return t;
}

}  // namespace

extern "C" {

const char* fs_last_error(void) { return g_err.c_str(); }

uint64_t fs_launch_count(void) { return g_launches.load(); }

int32_t fs_dump_stride(const fs_model* m) {
  if (!m) return 0;
  return (int32_t)align_up(sizeof(fs_scenario_head) + 8 * (size_t)m->d.K, 8);
}

int fs_load_model(const fs_bounds* b, const float* slo, const float* demand, int32_t G, void* cuda_stream,
                  fs_model** out) {
  NvtxRange nvtx_range("fs_load_model");
  if (!out) return fail(FS_EINVAL, "out is NULL");
  if (!b) return fail(FS_EINVAL, "bounds is NULL");
  if (b->K < 1 || b->K > FS_MAX_CLASSES) return fail(FS_EINVAL, "K = %d outside [1, %d]", b->K, FS_MAX_CLASSES);
  if (b->B < 1 || b->B > FS_MAX_BINS) return fail(FS_EINVAL, "B = %d outside [1, %d]", b->B, FS_MAX_BINS);
  if (G < 1 || G > FS_MAX_GPUS) return fail(FS_EINVAL, "G = %d outside [1, %d]", G, FS_MAX_GPUS);
  const int K = b->K, B = b->B, cells = K * 4 * B;
  const long long theta_cap = (long long)K * ((G >> 0) + (G >> 1) + (G >> 2) + (G >> 3));
  if (theta_cap > FS_MAX_THRESHOLDS)
    return fail(FS_EINVAL, "K * sum floor(G/tau) = %lld exceeds %d", theta_cap, FS_MAX_THRESHOLDS);
  int rc = check_bounds4(b->cap_lo, b->cap_hi, b->tail_lo, b->tail_hi, cells);
  if (rc) return rc;
  if (b->revealed)
    for (int c = 0; c < cells; ++c)
      if (b->revealed[c] && (b->cap_lo[c] != b->cap_hi[c] || b->tail_lo[c] != b->tail_hi[c]))
        return fail(FS_EINVAL, "cell %d is revealed but its bounds are not collapsed (lo != hi)", c);
  if (!slo || !demand) return fail(FS_EINVAL, "slo / demand is NULL");
  for (int i = 0; i < K; ++i) {
    if (!std::isfinite(slo[i]) || !(slo[i] > 0.0f)) return fail(FS_EINVAL, "slo[%d] must be finite and > 0", i);
    if (!std::isfinite(demand[i]) || !(demand[i] > 0.0f)) return fail(FS_EINVAL, "demand[%d] must be finite and > 0", i);
  }
  int Q = 4096;
  if (b->quantile) {
    Q = b->Q;
    if (!is_pow2(Q) || Q < 4 || Q > (1 << 24)) return fail(FS_EINVAL, "Q = %d must be a power of two in [4, 2^24]", Q);
    for (int k = 0; k < Q; ++k) {
      const float v = b->quantile[k];
      if (!(v >= 0.0f && v <= 1.0f)) return fail(FS_EINVAL, "quantile[%d] = %g outside [0, 1]", k, (double)v);
      if (k && v < b->quantile[k - 1]) return fail(FS_EINVAL, "quantile table decreases at %d", k);
    }
  }

  fs_model* m = new (std::nothrow) fs_model();
  if (!m) return fail(FS_ENOMEM, "host allocation");
  m->stream = (cudaStream_t)cuda_stream;
  cudaError_t e = cudaGetDevice(&m->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&m->sm_count, cudaDevAttrMultiProcessorCount, m->device);
  if (e != cudaSuccess) {
    delete m;
    return cuda_fail(e, "device query");
  }
  Dims& d = m->d;
  d.K = K;
  d.B = B;
  d.G = G;
  d.Q = Q;
  d.cells = cells;
  d.K4 = 4 * K;
  d.theta_cap = (int)theta_cap;
  d.lcap = 4;
  while (d.lcap < d.theta_cap + 1) d.lcap <<= 1;
  d.slot_floats = kTableHeader + 3 * d.lcap;

  // fixed device state, one allocation carved into 256-byte aligned pieces
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t o_lam = take(4 * K), o_slo = take(8 * K), o_qn = take(4 * (size_t)Q);
  const size_t o_bounds = take(16 * (size_t)cells), o_rev = take(cells);
  const size_t o_theta = take(8 * (size_t)d.theta_cap), o_nth = take(8);
  const size_t o_rowc = take(8 * (size_t)d.K4), o_rowb = take(8 * (size_t)d.K4);
  const size_t o_base = take(2 * sizeof(fs_allocation)), o_status = take(4), o_work = take(32);
  const size_t o_rtab = take(8 * (size_t)kRowTabMax);
  rc = m->fixed.ensure(off, "model state");
  if (rc) {
    delete m;
    return rc;
  }
  char* base = (char*)m->fixed.p;
  Set& s = m->set;
  s.d = d;
  s.P = 1;
  s.lam = (const float*)(base + o_lam);
  s.slo = (const float*)(base + o_slo);  // then the floors, zeroed below: no critical class
  s.qn = (const float*)(base + o_qn);
  s.bounds = (float*)(base + o_bounds);
  s.revealed = (uint8_t*)(base + o_rev);
  s.theta = (float*)(base + o_theta);
  s.ntheta = (int*)(base + o_nth);
  s.rowC = (float*)(base + o_rowc);
  s.rowB = (int*)(base + o_rowb);
  s.base = (fs_allocation*)(base + o_base);
  s.status = (uint32_t*)(base + o_status);
  s.work = (unsigned long long*)(base + o_work);
  s.skip = nullptr;
  s.rtab = (int*)(base + o_rtab);

  m->h_lam.assign(demand, demand + K);
  m->h_slo.assign(slo, slo + K);
  m->h_dlt.assign(K, 0.0f);
  m->h_bounds.resize(4 * (size_t)cells);
  const float* src[4] = {b->cap_lo, b->cap_hi, b->tail_lo, b->tail_hi};
  for (int r = 0; r < 4; ++r)
    for (int c = 0; c < cells; ++c) m->h_bounds[(size_t)r * cells + c] = canon(src[r][c]);
  m->h_revealed.assign(cells, 0);
  if (b->revealed)
    for (int c = 0; c < cells; ++c) m->h_revealed[c] = b->revealed[c] ? 1 : 0;

  auto bail = [&](int code) {
    fs_free_model(m);
    return code;
  };
  e = cudaMemsetAsync(m->fixed.p, 0, off, m->stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync((void*)s.lam, demand, 4 * K, cudaMemcpyHostToDevice, m->stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync((void*)s.slo, slo, 4 * K, cudaMemcpyHostToDevice, m->stream);
  if (e == cudaSuccess) {
    if (b->quantile) e = cudaMemcpyAsync((void*)s.qn, b->quantile, 4 * (size_t)Q, cudaMemcpyHostToDevice, m->stream);
    else e = launch_qtable((float*)s.qn, Q, m->stream);
  }
  if (e != cudaSuccess) return bail(cuda_fail(e, "model upload"));
  rc = stage_bounds(m);
  if (rc == FS_OK) rc = flush_bounds(m, m->stream);
  if (rc) return bail(rc);
  *out = m;
  return FS_OK;
}

int fs_update_bounds(fs_model* m, const float* cap_lo, const float* cap_hi, const float* tail_lo,
                     const float* tail_hi) {
  NvtxRange nvtx_range("fs_update_bounds");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  const int cells = m->d.cells;
  int rc = check_bounds4(cap_lo, cap_hi, tail_lo, tail_hi, cells);
  if (rc) return rc;
  const float* src[4] = {cap_lo, cap_hi, tail_lo, tail_hi};
  for (int r = 0; r < 4; ++r)
    for (int c = 0; c < cells; ++c) m->h_bounds[(size_t)r * cells + c] = canon(src[r][c]);
  return stage_bounds(m);
}

int fs_set_floors(fs_model* m, const float* floor) {
  NvtxRange nvtx_range("fs_set_floors");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  const int K = m->d.K;
  std::vector<float> v(K, 0.0f);
  if (floor)
    for (int i = 0; i < K; ++i) {
      if (!(floor[i] >= 0.0f && floor[i] <= 1.0f)) return fail(FS_EINVAL, "floor[%d] = %g outside [0, 1]", i, (double)floor[i]);
      v[i] = canon(floor[i]);
    }
  m->h_dlt = v;
  // a small copy, finished before the call returns: every later call on any
  // stream sees the new floors (they follow the SLOs on the device)
  FS_CUDA(cudaMemcpyAsync((void*)(m->set.slo + K), m->h_dlt.data(), 4 * (size_t)K, cudaMemcpyHostToDevice,
                          m->stream),
          "upload floors");
  FS_CUDA(cudaStreamSynchronize(m->stream), "upload floors");
  m->lc.floors = std::any_of(v.begin(), v.end(), [](float x) { return x > 0.0f; }) ? 1 : 0;
  return FS_OK;
}

int fs_score_candidates(fs_model* m, const fs_samples* smp, double* gap_out, double* score_out, float* gamma_t,
                        int32_t* best, int64_t* sum_eo, void* dump_dev) {
  NvtxRange nvtx_range("fs_score_candidates");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  int rc = check_samples(m, smp, true);
  if (rc) return rc;
  const int n = smp->n_cand;
  if ((rc = ensure_items(m, n, smp->O))) return rc;
  // One mapped page-locked block carries the call's host data both ways: the
  // kernels read the candidate ids from it and write gap, score, gamma_t, best
  // and the status word into it (k_finalize copies the status word), so no
  // copy engine sits before the first kernel or after the last one.
  const size_t nn = (size_t)std::max(n, 1);
  const size_t out_bytes = align_up(16 * nn + 36, 16);
  if ((rc = m->h_out.ensure(out_bytes + 4 * nn, "host staging"))) return rc;
  char* h = static_cast<char*>(m->h_out.p);
  char* hd = static_cast<char*>(m->h_out.dev);
  if (n > 0) std::memcpy(h + out_bytes, smp->cand, 4 * (size_t)n);
  double* d_gap = reinterpret_cast<double*>(hd);
  double* d_score = d_gap + nn;
  float* d_gt = reinterpret_cast<float*>(d_score + nn);
  int32_t* d_best = reinterpret_cast<int32_t*>(d_gt + 4);
  uint32_t* d_st = reinterpret_cast<uint32_t*>(d_best + 4);
  cudaStream_t s = m->stream;
  // freshly staged bounds are read where they are (their device copy waits
  // for the next call that needs it)
  Set set = m->set;
  if (m->staged) set.bounds = static_cast<float*>(m->h_up.dev);
  rc = run_score(m, set, smp, reinterpret_cast<const int32_t*>(hd + out_bytes), d_gap, d_score, d_gt, d_best,
                 dump_dev, s, d_st);
  if (rc) return rc;
  if (sum_eo && n)
    FS_CUDA(cudaMemcpyAsync(sum_eo, m->sums.p, 8 * (size_t)n * smp->O, cudaMemcpyDeviceToHost, s), "read sums");
  FS_CUDA(cudaStreamSynchronize(s), "synchronize");
  uint32_t st;
  std::memcpy(&st, h + 16 * nn + 32, 4);
  if (st) return status_error(m, st);
  if (gap_out && n) std::memcpy(gap_out, h, 8 * (size_t)n);
  if (score_out && n) std::memcpy(score_out, h + 8 * nn, 8 * (size_t)n);
  if (gamma_t) std::memcpy(gamma_t, h + 16 * nn, 4);
  if (best) std::memcpy(best, h + 16 * nn + 16, 4);
  return FS_OK;
}

int fs_score_candidates_async(fs_model* m, const fs_samples* smp, double* gap_dev, double* score_dev,
                              float* gamma_t_dev, int32_t* best_dev, int64_t* sum_eo_dev, void* dump_dev,
                              void* cuda_stream) {
  NvtxRange nvtx_range("fs_score_candidates_async");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  int rc = check_samples(m, smp, false);
  if (rc) return rc;
  const int n = smp->n_cand;
  if ((rc = ensure_items(m, n, smp->O))) return rc;
  cudaStream_t s = (cudaStream_t)cuda_stream;
  if ((rc = flush_bounds(m, s))) return rc;
  rc = run_score(m, m->set, smp, smp->cand, gap_dev, score_dev, gamma_t_dev, best_dev, dump_dev, s);
  if (rc) return rc;
  if (sum_eo_dev && n)
    FS_CUDA(cudaMemcpyAsync(sum_eo_dev, m->sums.p, 8 * (size_t)n * smp->O, cudaMemcpyDeviceToDevice, s),
            "copy sums");
  return FS_OK;
}

int fs_solve(fs_model* m, const float* cap, const float* tail, fs_allocation* out) {
  NvtxRange nvtx_range("fs_solve");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (!out) return fail(FS_EINVAL, "out is NULL");
  const int cells = m->d.cells;
  int rc;
  if ((rc = check_cells(cap, cells, "cap")) || (rc = check_cells(tail, cells, "tail"))) return rc;
  if ((rc = m->real.ensure(8 * (size_t)cells + 256 + sizeof(fs_allocation), "realisation"))) return rc;
  float* d_cap = (float*)m->real.p;
  float* d_tail = d_cap + cells;
  fs_allocation* d_out = (fs_allocation*)((char*)m->real.p + align_up(8 * (size_t)cells, 256));
  cudaStream_t s = m->stream;
  FS_CUDA(cudaMemcpyAsync(d_cap, cap, 4 * (size_t)cells, cudaMemcpyHostToDevice, s), "upload cap");
  FS_CUDA(cudaMemcpyAsync(d_tail, tail, 4 * (size_t)cells, cudaMemcpyHostToDevice, s), "upload tail");
  FS_CUDA(launch_solve(m->set, 1, d_cap, d_tail, d_out, false, m->lc, s), "launch solve");
  if ((rc = solve_lex_pass(m, m->set, 1, d_cap, d_tail, d_out, s))) return rc;
  FS_CUDA(cudaMemcpyAsync(out, d_out, sizeof(fs_allocation), cudaMemcpyDeviceToHost, s), "read allocation");
  return read_status(m, s);
}

int fs_solve_batch(fs_model* m, int32_t n, const float* cap_dev, const float* tail_dev, fs_allocation* out_dev,
                   void* cuda_stream) {
  NvtxRange nvtx_range("fs_solve_batch");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (n < 0) return fail(FS_EINVAL, "n < 0");
  if (n == 0) return FS_OK;
  if (!cap_dev || !tail_dev || !out_dev) return fail(FS_EINVAL, "NULL device pointer");
  int rc = flush_bounds(m, (cudaStream_t)cuda_stream);
  if (rc) return rc;
  FS_CUDA(launch_solve(m->set, n, cap_dev, tail_dev, out_dev, false, m->lc, (cudaStream_t)cuda_stream),
          "launch solve");
  return solve_lex_pass(m, m->set, n, cap_dev, tail_dev, out_dev, (cudaStream_t)cuda_stream);
}

int fs_solve_bounds(fs_model* m, fs_allocation* minus, fs_allocation* plus, float* gamma_t) {
  NvtxRange nvtx_range("fs_solve_bounds");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  cudaStream_t s = m->stream;
  int rc0 = flush_bounds(m, s);
  if (rc0) return rc0;
  FS_CUDA(launch_solve(m->set, 2, nullptr, nullptr, nullptr, true, m->lc, s), "launch solve");
  if ((rc0 = solve_lex_pass(m, m->set, 2, nullptr, nullptr, nullptr, s))) return rc0;
  fs_allocation h[2];
  FS_CUDA(cudaMemcpyAsync(h, m->set.base, sizeof h, cudaMemcpyDeviceToHost, s), "read allocations");
  int rc = read_status(m, s);
  if (rc) return rc;
  if (minus) *minus = h[0];
  if (plus) *plus = h[1];
  if (gamma_t) *gamma_t = h[1].t_star - h[0].t_star;
  return FS_OK;
}

int fs_reveal(fs_model* m, int32_t cell, float cap, float tail) {
  NvtxRange nvtx_range("fs_reveal");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (cell < 0 || cell >= m->d.cells) return fail(FS_EINVAL, "cell %d out of range", cell);
  if (!std::isfinite(cap) || cap < 0.0f || !std::isfinite(tail) || tail < 0.0f)
    return fail(FS_EINVAL, "measured values must be finite and >= 0");
  refit_cell(m->h_bounds.data(), m->d.cells, m->d.B, m->set.prior, cell, canon(cap), canon(tail));
  m->h_revealed[cell] = 1;
  return stage_bounds(m);
}

int fs_set_prior(fs_model* m, int32_t prior) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (prior != FS_PRIOR_REVEALED && prior != FS_PRIOR_MONOTONE) return fail(FS_EINVAL, "prior %d is not 0 or 1", prior);
  m->set.prior = prior;
  return FS_OK;
}

int fs_get_state(const fs_model* m, float* cap_lo, float* cap_hi, float* tail_lo, float* tail_hi,
                 uint8_t* revealed) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  const size_t cells = (size_t)m->d.cells;
  float* dst[4] = {cap_lo, cap_hi, tail_lo, tail_hi};
  for (int r = 0; r < 4; ++r)
    if (dst[r]) std::memcpy(dst[r], m->h_bounds.data() + (size_t)r * cells, 4 * cells);
  if (revealed) std::memcpy(revealed, m->h_revealed.data(), cells);
  return FS_OK;
}

int fs_certificate(fs_model* m, float eps, int32_t* state, float* gamma_t) {
  NvtxRange nvtx_range("fs_certificate");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (!state) return fail(FS_EINVAL, "state is NULL");
  if (std::isnan(eps)) return fail(FS_EINVAL, "eps is NaN");
  fs_allocation am, ap;
  float gt;
  int rc = fs_solve_bounds(m, &am, &ap, &gt);
  if (rc) return rc;
  bool known = true;
  for (int i = 0; i < m->d.K; ++i) {
    if (am.replicas[i] <= 0) continue;
    int j = 0;
    while (j < kT && (1 << j) != am.tp[i]) ++j;
    if (!m->h_revealed[(size_t)(i * 4 + j) * m->d.B + am.bin[i]]) known = false;
  }
  // under the lexicographic objective the gap is stage-wise (Section 4.2):
  // the goodput gap |GP+ - GP-| / sum lambda must be within eps as well
  bool gp_ok = true;
  if (m->objective == FS_OBJECTIVE_LEXICOGRAPHIC)
    gp_ok = std::fabs(ap.goodput - am.goodput) / demand_sum(m) <= (double)eps;
  if (!ap.floors_met) *state = 2;
  else *state = (am.floors_met && gt <= eps && known && gp_ok) ? 1 : 0;
  if (gamma_t) *gamma_t = gt;
  return FS_OK;
}

int fs_set_objective(fs_model* m, int32_t objective) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (objective != FS_OBJECTIVE_MAXMIN && objective != FS_OBJECTIVE_LEXICOGRAPHIC)
    return fail(FS_EINVAL, "objective %d is not 0 or 1", objective);
  if (objective == FS_OBJECTIVE_LEXICOGRAPHIC && lex_scratch_cells(m->d) * kLexCellBytes > (64u << 20))
    return fail(FS_EINVAL, "the lexicographic objective needs (K + 1)(G + 1) <= 4 Mi cells");
  m->objective = objective;
  return FS_OK;
}

int fs_score_goodput(fs_model* m, const fs_samples* smp, double* gap_out, double* score_out, double* gamma_gp,
                     int32_t* best, int64_t* sum_eo) {
  NvtxRange nvtx_range("fs_score_goodput");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  int rc = check_samples(m, smp, true);
  if (rc) return rc;
  const double lam_sum = demand_sum(m);
  if (!(lam_sum <= 1048576.0)) return fail(FS_EINVAL, "the goodput stage needs sum lambda <= 2^20 req/s");
  if (m->d.G > 1024) return fail(FS_EINVAL, "the goodput stage needs G <= 1024");
  if (lex_scratch_cells(m->d) * kLexCellBytes > (64u << 20)) return fail(FS_EINVAL, "(K + 1)(G + 1) too large");
  const int n = smp->n_cand;
  if ((rc = ensure_items(m, n, smp->O))) return rc;
  cudaStream_t s = m->stream;
  if ((rc = flush_bounds(m, s))) return rc;
  // as in fs_score_candidates, one mapped page-locked block carries the
  // candidate ids in and gap, score, gamma, best and the status word out
  const size_t nn = (size_t)std::max(n, 1);
  const size_t out_bytes = align_up(16 * nn + 16, 16);
  if ((rc = m->h_out.ensure(out_bytes + 4 * nn, "host staging"))) return rc;
  char* h = static_cast<char*>(m->h_out.p);
  char* hd = static_cast<char*>(m->h_out.dev);
  if (n > 0) std::memcpy(h + out_bytes, smp->cand, 4 * (size_t)n);
  double* d_gap = reinterpret_cast<double*>(hd);
  double* d_score = d_gap + nn;
  double* d_gamma = reinterpret_cast<double*>(hd + 16 * nn);
  int32_t* d_best = reinterpret_cast<int32_t*>(hd + 16 * nn + 8);
  uint32_t* d_st = reinterpret_cast<uint32_t*>(hd + 16 * nn + 12);
  Items it{};
  it.n = n;
  it.cell = reinterpret_cast<const int32_t*>(hd + out_bytes);
  const Plan pl = make_plan(m, smp, n);
  if (goodput_threads(m->d, pl, m->set.prior == 1, nullptr) == 0)
    return fail(FS_EINVAL, "the goodput stage needs Q / O <= 2048 under the monotone prior, 4096 otherwise");
  const int saved = m->objective;
  m->objective = FS_OBJECTIVE_LEXICOGRAPHIC;  // the base solves to tier 4 (their goodput)
  FS_CUDA(launch_solve(m->set, 2, nullptr, nullptr, nullptr, true, m->lc, s), "launch solve");
  rc = solve_lex_pass(m, m->set, 2, nullptr, nullptr, nullptr, s);
  m->objective = saved;
  if (rc) return rc;
  uint64_t* sums = static_cast<uint64_t*>(m->sums.p);
  FS_CUDA(launch_prep(m->set, it, pl, static_cast<float*>(m->tables.p), sums, false, m->sm_count, m->lc, s),
          "launch prep");
  FS_CUDA(launch_score_goodput(m->set, it, pl, static_cast<const float*>(m->tables.p), sums, m->lc.floors,
                               m->sm_count, s),
          "launch goodput scorer");
  FS_CUDA(launch_finalize_goodput(m->set, it, pl, sums, lam_sum, d_gap, d_score, d_gamma, d_best, d_st, s),
          "launch goodput reduction");
  if (sum_eo && n)
    FS_CUDA(cudaMemcpyAsync(sum_eo, sums, 8 * (size_t)n * smp->O, cudaMemcpyDeviceToHost, s), "read sums");
  FS_CUDA(cudaStreamSynchronize(s), "synchronize");
  uint32_t st;
  std::memcpy(&st, h + 16 * nn + 12, 4);
  if (st) return status_error(m, st);
  if (gap_out && n) std::memcpy(gap_out, h, 8 * (size_t)n);
  if (score_out && n) std::memcpy(score_out, h + 8 * nn, 8 * (size_t)n);
  if (gamma_gp) std::memcpy(gamma_gp, h + 16 * nn, 8);
  if (best) std::memcpy(best, h + 16 * nn + 8, 4);
  return FS_OK;
}

int fs_replay(fs_model* m, const fs_replay_spec* sp, int32_t* rounds, int32_t* state, double* gpu_seconds,
              int32_t* reveal_order, float* gamma_trace, fs_allocation* final_minus) {
  NvtxRange nvtx_range("fs_replay");
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (!sp) return fail(FS_EINVAL, "spec is NULL");
  const Dims d = m->d;
  const int P = sp->n_streams, cells = d.cells;
  if (P < 1 || P > 65536) return fail(FS_EINVAL, "n_streams = %d outside [1, 65536]", P);
  if (sp->r0 < 0 || sp->r0 > cells) return fail(FS_EINVAL, "r0 = %d outside [0, cells]", sp->r0);
  if (sp->max_rounds < 0 || sp->max_rounds > cells) return fail(FS_EINVAL, "max_rounds outside [0, cells]");
  if (std::isnan(sp->eps)) return fail(FS_EINVAL, "eps is NaN");
  if (sp->policy < 0 || sp->policy > 1) return fail(FS_EINVAL, "policy = %d is not 0 or 1", sp->policy);
  if (!sp->truth_cap || !sp->truth_tail || !sp->perm) return fail(FS_EINVAL, "NULL truth / perm");
  fs_samples probe{sp->seed, 0, 0, 0, sp->O, sp->S, 0, nullptr};
  int rc = check_samples(m, &probe, false);
  if (rc) return rc;
  if ((rc = check_cells(sp->truth_cap, P * cells, "truth_cap")) || (rc = check_cells(sp->truth_tail, P * cells, "truth_tail")))
    return rc;
  std::vector<char> seen(cells);
  for (int k = 0; k < P; ++k) {
    std::fill(seen.begin(), seen.end(), 0);
    for (int q = 0; q < cells; ++q) {
      const int c = sp->perm[(size_t)k * cells + q];
      if (c < 0 || c >= cells || seen[c]) return fail(FS_EINVAL, "perm[%d] is not a permutation of the cells", k);
      seen[c] = 1;
    }
  }

  // device state of P problems
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t o_bounds = take(16 * (size_t)P * cells), o_rev = take((size_t)P * cells);
  const size_t o_theta = take(8 * (size_t)P * d.theta_cap), o_nth = take(8 * (size_t)P);
  const size_t o_rowc = take(8 * (size_t)P * d.K4), o_rowb = take(8 * (size_t)P * d.K4);
  const size_t o_base = take(2 * (size_t)P * sizeof(fs_allocation));
  const size_t o_truth = take(8 * (size_t)P * cells), o_perm = take(4 * (size_t)P * cells);
  const size_t o_rounds = take(4 * (size_t)P), o_state = take(4 * (size_t)P), o_gs = take(8 * (size_t)P);
  const size_t o_order = take(4 * (size_t)P * cells), o_nrev = take(4 * (size_t)P);
  const size_t o_trace = take(4 * (size_t)P * (sp->max_rounds + 1));
  const size_t o_final = take((size_t)P * sizeof(fs_allocation)), o_active = take(4 * (size_t)P), o_nact = take(4);
  const size_t o_ip = take(4 * (size_t)P * cells), o_ic = take(4 * (size_t)P * cells);
  const size_t o_rtab = take(8 * (size_t)P * kRowTabMax);
  const size_t o_prior = take(16 * (size_t)cells);
  Buf& all = m->replay;
  if ((rc = all.ensure(off, "replay state"))) return rc;
  char* base = (char*)all.p;
  Set set = m->set;
  set.P = P;
  set.bounds = (float*)(base + o_bounds);
  set.revealed = (uint8_t*)(base + o_rev);
  set.theta = (float*)(base + o_theta);
  set.ntheta = (int*)(base + o_nth);
  set.rowC = (float*)(base + o_rowc);
  set.rowB = (int*)(base + o_rowb);
  set.base = (fs_allocation*)(base + o_base);
  set.rtab = (int*)(base + o_rtab);
  ReplayState rs{};
  rs.truth = (const float*)(base + o_truth);
  rs.perm = (const int*)(base + o_perm);
  rs.rounds = (int*)(base + o_rounds);
  rs.state = (int*)(base + o_state);
  rs.gpu_seconds = (double*)(base + o_gs);
  rs.reveal_order = (int*)(base + o_order);
  rs.n_revealed = (int*)(base + o_nrev);
  rs.gamma_trace = (float*)(base + o_trace);
  rs.final_minus = (fs_allocation*)(base + o_final);
  rs.active = (int*)(base + o_active);
  rs.n_active = (int*)(base + o_nact);
  rs.item_p = (int*)(base + o_ip);
  rs.item_cell = (int*)(base + o_ic);
  rs.max_rounds = sp->max_rounds;
  rs.eps = sp->eps;
  set.skip = rs.state;

  cudaStream_t s = m->stream;
  auto run = [&]() -> int {
    FS_CUDA(cudaMemsetAsync(all.p, 0, off, s), "clear replay state");
    // the prior once; the init kernel gives every stream its copy
    float* prior = (float*)(base + o_prior);
    FS_CUDA(cudaMemcpyAsync(prior, m->h_bounds.data(), 16 * (size_t)cells, cudaMemcpyHostToDevice, s),
            "upload prior");
    std::vector<float> truth(2 * (size_t)P * cells);
    for (int k = 0; k < P; ++k) {
      std::memcpy(&truth[(2 * (size_t)k) * cells], sp->truth_cap + (size_t)k * cells, 4 * (size_t)cells);
      std::memcpy(&truth[(2 * (size_t)k + 1) * cells], sp->truth_tail + (size_t)k * cells, 4 * (size_t)cells);
    }
    for (auto& v : truth) v = canon(v);
    FS_CUDA(cudaMemcpyAsync((void*)rs.truth, truth.data(), 4 * truth.size(), cudaMemcpyHostToDevice, s), "upload truth");
    FS_CUDA(cudaMemcpyAsync((void*)rs.perm, sp->perm, 4 * (size_t)P * cells, cudaMemcpyHostToDevice, s), "upload perm");
    FS_CUDA(launch_replay_init(set, rs, prior, sp->r0, s), "launch replay init");
    const int rc_sync = read_status(m, s);  // truth buffer must outlive the copy
    if (rc_sync) return rc_sync;
    for (int r = 0; r <= sp->max_rounds; ++r) {
      FS_CUDA(launch_solve(set, 2 * P, nullptr, nullptr, nullptr, true, m->lc, s), "launch solve");
      FS_CUDA(cudaMemsetAsync(rs.n_active, 0, 4, s), "clear active");
      const int per = cells - sp->r0 - r;  // candidates of each running stream this round
      // the certificate, and the running streams' candidate lists (scored reveals)
      FS_CUDA(launch_replay_certify(set, rs, r, sp->policy == 0 ? per : 0, s), "launch certify");
      int n_active = 0;
      FS_CUDA(cudaMemcpyAsync(&n_active, rs.n_active, 4, cudaMemcpyDeviceToHost, s), "read active");
      FS_CUDA(cudaStreamSynchronize(s), "round sync");
      if (n_active == 0) break;
      if (per <= 0) break;
      if (sp->policy == 1) {
        FS_CUDA(launch_replay_next(set, rs, n_active, s), "launch reveal");
        continue;
      }
      const int n_items = n_active * per;
      int rc2 = ensure_items(m, n_items, sp->O);
      if (rc2) return rc2;
      Items it{};
      it.n = n_items;
      it.p = rs.item_p;
      it.cell = rs.item_cell;
      it.off = nullptr;
      fs_samples smp{sp->seed, 0, (uint32_t)r, n_items, sp->O, sp->S, 0, nullptr};
      const Plan pl = make_plan(m, &smp, n_items);
      FS_CUDA(launch_prep(set, it, pl, (float*)m->tables.p, (uint64_t*)m->sums.p, false, m->sm_count, m->lc, s),
              "launch prep");
      FS_CUDA(launch_score(set, it, pl, (const float*)m->tables.p, (uint64_t*)m->sums.p, nullptr, 0, m->sm_count,
                           m->lc, s),
              "launch score");
      FS_CUDA(launch_replay_reveal(set, rs, it, pl, (const uint64_t*)m->sums.p, n_active, s), "launch reveal");
    }
    if (rounds) FS_CUDA(cudaMemcpyAsync(rounds, rs.rounds, 4 * (size_t)P, cudaMemcpyDeviceToHost, s), "read rounds");
    if (state) FS_CUDA(cudaMemcpyAsync(state, rs.state, 4 * (size_t)P, cudaMemcpyDeviceToHost, s), "read state");
    if (gpu_seconds)
      FS_CUDA(cudaMemcpyAsync(gpu_seconds, rs.gpu_seconds, 8 * (size_t)P, cudaMemcpyDeviceToHost, s), "read gpu-s");
    if (reveal_order)
      FS_CUDA(cudaMemcpyAsync(reveal_order, rs.reveal_order, 4 * (size_t)P * cells, cudaMemcpyDeviceToHost, s),
              "read order");
    if (gamma_trace)
      FS_CUDA(cudaMemcpyAsync(gamma_trace, rs.gamma_trace, 4 * (size_t)P * (sp->max_rounds + 1),
                              cudaMemcpyDeviceToHost, s),
              "read trace");
    if (final_minus)
      FS_CUDA(cudaMemcpyAsync(final_minus, rs.final_minus, sizeof(fs_allocation) * (size_t)P, cudaMemcpyDeviceToHost,
                              s),
              "read allocations");
    return read_status(m, s);
  };
  rc = run();
  cudaStreamSynchronize(s);
  return rc;
}

int fs_check(fs_model* m, void* cuda_stream) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  return read_status(m, cuda_stream ? (cudaStream_t)cuda_stream : m->stream);
}

// The work counts (work[2..3]) of the model, zeroed in stream order.
static int zero_entry_count(fs_model* m) {
  FS_CUDA(cudaMemsetAsync(m->set.work + 2, 0, 16, m->stream), "zero the entry count");
  FS_CUDA(cudaStreamSynchronize(m->stream), "zero the entry count");
  return FS_OK;
}

int fs_timing_enable(fs_model* m, int32_t on) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (on < 0 || on > 2) return fail(FS_EINVAL, "timing mode %d not in {0, 1, 2}", on);
  m->timing = on;
  m->ev_used = 0;
  return zero_entry_count(m);
}

int fs_timing_read(fs_model* m, double* kernel_ms, int32_t* launches, double* phase_ms, uint64_t* work_counts) {
  if (!m) return fail(FS_EINVAL, "model is NULL");
  if (work_counts) {
    FS_CUDA(cudaDeviceSynchronize(), "wait for the scoring calls");
    FS_CUDA(cudaMemcpy(work_counts, m->set.work + 2, 16, cudaMemcpyDeviceToHost), "read the work counts");
    int rc = zero_entry_count(m);
    if (rc) return rc;
  }
  double total = 0.0, ph[4] = {0.0, 0.0, 0.0, 0.0};
  const size_t n = m->ev_used / 5;
  for (size_t k = 0; k < n; ++k) {
    cudaEvent_t* e = &m->ev[5 * k];
    FS_CUDA(cudaEventSynchronize(e[3]), "wait timing event");
    float ms = 0.0f;
    FS_CUDA(cudaEventElapsedTime(&ms, e[2], e[3]), "elapsed time");
    total += ms;
    if (m->timing == 2) {
      FS_CUDA(cudaEventSynchronize(e[4]), "wait timing event");
      for (int q = 0; q < 4; ++q) {
        FS_CUDA(cudaEventElapsedTime(&ms, e[q], e[q + 1]), "elapsed time");
        ph[q] += ms;
      }
    }
  }
  m->ev_used = 0;
  if (kernel_ms) *kernel_ms = total;
  if (launches) *launches = (int32_t)n;
  if (phase_ms)
    for (int q = 0; q < 4; ++q) phase_ms[q] = ph[q];
  return FS_OK;
}

int fs_draw_floor(int32_t mode, int32_t w, int64_t calls, int32_t reps, double* ms, int64_t* calls_done) {
  if (mode != 0 && mode != 1) return fail(FS_EINVAL, "fs_draw_floor: mode must be 0 or 1");
  if (w < 0 || w > 12) return fail(FS_EINVAL, "fs_draw_floor: w must be in [0, 12]");
  if (calls < 1 || calls > (1LL << 36)) return fail(FS_EINVAL, "fs_draw_floor: calls must be in [1, 2^36]");
  if (reps < 1 || reps > 1000) return fail(FS_EINVAL, "fs_draw_floor: reps must be in [1, 1000]");
  if (!ms || !calls_done) return fail(FS_EINVAL, "fs_draw_floor: null output");
  int dev = 0, sms = 0;
  FS_CUDA(cudaGetDevice(&dev), "current device");
  FS_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev), "SM count");
  long long done = 0;
  const cudaError_t e = draw_floor(mode, w, calls, reps, sms, ms, &done);
  if (e == cudaErrorInvalidValue) return fail(FS_EINVAL, "fs_draw_floor: too many calls per thread");
  if (e != cudaSuccess) return cuda_fail(e, "draw floor");
  *calls_done = done;
  return FS_OK;
}

int fs_watchdog_selftest(int64_t timeout_ns) {
  const int64_t t = std::min<int64_t>(std::max<int64_t>(timeout_ns, 1000000), 5000000000LL);
  uint32_t* st = nullptr;
  FS_CUDA(cudaMalloc(&st, 4), "watchdog status");
  cudaError_t e = cudaMemset(st, 0, 4);
  if (e == cudaSuccess) e = launch_watchdog(st, (uint64_t)t, nullptr);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  uint32_t v = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&v, st, 4, cudaMemcpyDeviceToHost);
  cudaFree(st);
  if (e != cudaSuccess) return cuda_fail(e, "watchdog self-test");
  if (v & ST_TIMEOUT) return fail(FS_ETIMEOUT, "watchdog: the barrier wait gave up after %lld ns", (long long)t);
  return fail(FS_EDEVICE, "watchdog: the wait did not report a timeout (status 0x%x)", v);
}

void fs_free_model(fs_model* m) {
  if (!m) return;
  if (m->stream) cudaStreamSynchronize(m->stream);
  else cudaDeviceSynchronize();
  m->fixed.release();
  m->cand.release();
  m->tables.release();
  m->sums.release();
  m->outs.release();
  m->real.release();
  m->lex.release();
  m->replay.release();
  for (cudaEvent_t e : m->ev) cudaEventDestroy(e);
  if (m->up_done) cudaEventDestroy(m->up_done);
  m->h_up.release();
  m->h_out.release();
  delete m;
}

}  // extern "C"
