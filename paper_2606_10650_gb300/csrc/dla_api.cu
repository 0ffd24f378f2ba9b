// dla_api.cu -- extern "C" entry points of libdla.so (see include/dla.h).
//
// Host logic only: argument checks, workspace layout, the round schedule of
// the forward pass and the kernel launches.  Every compute step runs in the
// kernels of dla_scan.cu / dla_readout_*.cu / dla_decode.cu.
#include <cuda.h>
#include <math.h>
#include <algorithm>
#include <mutex>
#include <stdarg.h>
#include <vector>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "dla.h"
#include "dla_kernels.h"

namespace {

thread_local char g_err[512] = "";

dla_status fail(dla_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

dla_status ok() {
  g_err[0] = '\0';
  return DLA_OK;
}

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

struct CacheLayout {
  size_t states, slot, n, ibar, m, total;
};

CacheLayout cache_layout(int B, int H, int C, int dk, int dv) {
  CacheLayout L;
  const size_t BH = (size_t)B * H;
  size_t off = 0;
  L.states = off; off = align256(off + BH * C * (size_t)dk * dv * sizeof(float));
  L.slot = off;   off = align256(off + BH * C * sizeof(int32_t));
  L.n = off;      off = align256(off + BH * C * sizeof(int32_t));
  L.ibar = off;   off = align256(off + BH * C * sizeof(double));
  L.m = off;      off = align256(off + BH * sizeof(int32_t));
  L.total = off;
  return L;
}

// The read-out kernel of a configuration: bf16 inputs with d = 128 run on the
// tensor cores (128-token intervals, fp16 snapshots with a power-of-two scale
// per entry); everything else on CUDA cores (64-token intervals, fp32 snapshots).
bool use_tc(dla_dtype in_dtype, int d) { return in_dtype == DLA_BF16 && d == 128; }
int readout_interval(dla_dtype in_dtype, int d) {
  return use_tc(in_dtype, d) ? dla::kReadoutTcInterval : dla::kReadoutSimtInterval;
}

// Workspace plan of a forward call.  The read-out needs, for every interval,
// the list of cache entries at its start (snapshot lists) and a pool holding
// those entries' states.  Persistent mode: one append-only pool for the whole
// sequence, so rounds continue it and a scan never waits for a read-out.
// Reset mode (small workspaces): each round restarts a pool of its own, two
// pools alternate, and a round copies the live states into its pool first.
constexpr int kInputPieces = 16;  // pieces of inputs streamed in from host memory (dla_forward_host)
constexpr int kOutPieces = 16;    // pieces of the output copied back while the read-out runs

struct FwdPlan {
  int interval;      // tokens per snapshot interval
  int nsnap_total;   // intervals over the whole sequence
  int R;             // intervals per round
  int rounds;
  int persistent;
  int nbuf;          // pools (1 persistent, 2 reset with several rounds)
  int pool_cap;      // pool entries per stream, per pool
  size_t off_status, off_rows, off_bnd, off_mlog, off_cache, off_lists_m0, off_lists_ids, off_pstate, off_nbound,
      off_gram, off_progress, off_pool, pool_bytes, pool_scale_off;
  int gram_chunks;   // chunks of the Gram pre-pass output (0: the scan forms its Gram entries itself)
  size_t total;
};

// Bytes per snapshot element: fp32 (CUDA-core read-out) or fp16 (tensor-core
// read-out: S / s in fp16 with s a power of two per entry, kept beside the
// entries).  A single bf16 rounding of the states (2^-9 relative) already
// reaches the 2e-2 output tolerance on coherent (regime) streams; fp16 keeps
// 2^-12, eight times less.
size_t pool_elt(dla_dtype in_dtype, int d) { return use_tc(in_dtype, d) ? 2 : 4; }

FwdPlan plan_for(int R, bool persistent, const dla_params* p, int B, int T, int H, int d, dla_dtype in_dtype,
                 bool with_output, bool need_trace, bool need_cache) {
  FwdPlan P;
  const size_t BH = (size_t)B * H;
  const int C = p->capacity;
  P.interval = readout_interval(in_dtype, d);
  P.nsnap_total = (T + P.interval - 1) / P.interval;
  P.R = R;
  P.rounds = (P.nsnap_total + R - 1) / R;
  P.persistent = persistent ? 1 : 0;
  const int per_snap = C < P.interval + 1 ? C : P.interval + 1;
  if (!with_output) {
    P.nbuf = 0;
    P.pool_cap = 0;
  } else if (persistent) {
    P.nbuf = 1;
    P.pool_cap = C + (P.nsnap_total - 1) * per_snap;
  } else {
    P.nbuf = P.rounds > 1 ? 2 : 1;
    P.pool_cap = C + (R - 1) * per_snap;
  }
  size_t off = 0;
  P.off_status = off;    off = align256(off + 256);
  // packed batches: each row's length and first token row (2 x B int32)
  P.off_rows = off;      off = align256(off + 2 * (size_t)B * sizeof(int32_t));
  P.off_bnd = off;       if (need_trace) off = align256(off + BH * T);
  P.off_mlog = off;      if (need_trace) off = align256(off + BH * T * sizeof(int32_t));
  P.off_cache = off;     if (need_cache) off = align256(off + cache_layout(B, H, C, d, d).total);
  P.off_lists_m0 = off;  if (with_output) off = align256(off + BH * P.nsnap_total * sizeof(int32_t));
  P.off_lists_ids = off; if (with_output) off = align256(off + BH * P.nsnap_total * C * sizeof(int32_t));
  P.off_pstate = off;    if (with_output) off = align256(off + (BH + BH * C) * sizeof(int32_t));
  // norm bounds of the live entries between rounds (tensor-core read-out: the scale of a snapshot)
  P.off_nbound = off;    if (with_output) off = align256(off + BH * C * sizeof(float));
  // Gram pre-pass output (bf16 inputs, calls with a read-out): kGramStride floats per 64-token chunk
  P.gram_chunks = (with_output && in_dtype == DLA_BF16) ? (T + dla::kScanL - 1) / dla::kScanL : 0;
  P.off_gram = off;      off = align256(off + BH * (size_t)P.gram_chunks * dla::kGramStride * 4);
  // scan progress per (stream, CTA), the count of started scan CTAs (concurrent read-out),
  // the count of input pieces streamed in by the host, and the Gram pre-pass's per-block
  // chunk counters (a pre-pass running beside the scan)
  P.off_progress = off;
  if (with_output) off = align256(off + (2 * BH + 2 + kOutPieces + BH * dla::kMaxGramBlk) * sizeof(int32_t));
  // a pool: its entries, then (tensor-core read-out) one scale per entry
  P.pool_scale_off = with_output ? align256(BH * (size_t)P.pool_cap * d * d * pool_elt(in_dtype, d)) : 0;
  P.pool_bytes = P.pool_scale_off +
                 ((with_output && use_tc(in_dtype, d)) ? align256(BH * (size_t)P.pool_cap * sizeof(float)) : 0);
  P.off_pool = off;      off += (size_t)P.nbuf * P.pool_bytes;
  P.total = off;
  return P;
}

// Interval counts of the rounds, in order.  Rounds of at most R intervals,
// balanced; with `taper` followed by rounds of R/2, R/4, R/8 intervals, so that
// the read-out left to run after the last scan launch is short.
std::vector<int> round_sizes(const FwdPlan& P, bool taper) {
  std::vector<int> out, tail;
  int left = P.nsnap_total;
  if (taper)
    for (int s = P.R / 2; s >= 1 && s >= P.R / 8 && left - s >= P.R; s /= 2) {
      tail.push_back(s);
      left -= s;
    }
  const int n = (left + P.R - 1) / P.R;
  for (int i = 0; i < n; ++i) out.push_back(left / n + (i < left % n ? 1 : 0));
  out.insert(out.end(), tail.begin(), tail.end());
  return out;
}

}  // namespace

namespace dla {
void finish_score_params(ScoreParams& sp) {
  float t = (float)sp.tau;
  if ((double)t < sp.tau) t = nextafterf(t, INFINITY);
  sp.tau_f = t;
  sp.eps_f = (float)sp.eps;
  sp.rms_eps_f = (float)sp.rms_eps;
}
}  // namespace dla

namespace {

// Schedule of the tensor-core forward pass (environment variable DLA_SCHEDULE,
// read at every call): "concurrent" (default) launches the scan once over the
// whole sequence, the Gram pre-pass and the read-out beside it, each waiting
// for the other side's progress; "rounds" launches the scan once per round and
// the round's read-out after it; "serial" runs the pre-pass, the whole scan and
// one read-out launch one after another, each kernel alone on the device (no
// kernel waits for another: for timing and profiling single kernels).  All
// compute the same results.
enum Schedule { kConcurrent, kRounds, kSerial };
// DLA_SCAN=tc (read at every call) selects the tcgen05 scan where it applies.
bool scan_tc_requested() {
  const char* v = getenv("DLA_SCAN");
  return v && strcmp(v, "tc") == 0;
}
Schedule schedule() {
  const char* v = getenv("DLA_SCHEDULE");
  if (v && strcmp(v, "rounds") == 0) return kRounds;
  if (v && strcmp(v, "serial") == 0) return kSerial;
  return kConcurrent;
}

constexpr int kTargetRounds = 8;  // rounds the read-out overlaps with the scan
constexpr int kMinFreeSms = 8;    // SMs the scan must leave free for the concurrent schedule
constexpr size_t kPreferredWorkspace = (size_t)16 << 30;  // 16 GiB of read-out staging

dla_status check_params(const dla_params* p) {
  if (!p) return fail(DLA_ERR_INVALID_ARG, "params is NULL");
  if (!isfinite(p->tau)) return fail(DLA_ERR_INVALID_ARG, "tau must be finite");
  if (!(p->eps >= 0.0) || !(p->rms_eps >= 0.0)) return fail(DLA_ERR_INVALID_ARG, "eps and rms_eps must be >= 0");
  if (p->capacity < 2) return fail(DLA_ERR_INVALID_ARG, "capacity must be >= 2 (Algorithm 2 merges a pair)");
  if (p->capacity > dla::kMaxCBig) return fail(DLA_ERR_UNSUPPORTED, "capacity %d > %d", p->capacity, dla::kMaxCBig);
  if (p->score_mode != 0 && p->score_mode != 1) return fail(DLA_ERR_INVALID_ARG, "score_mode must be 0 or 1");
  if (p->out_dtype != DLA_BF16 && p->out_dtype != DLA_F32) return fail(DLA_ERR_INVALID_ARG, "bad out_dtype");
  if (p->from_cache != 0 && p->from_cache != 1) return fail(DLA_ERR_INVALID_ARG, "from_cache must be 0 or 1");
  return DLA_OK;
}

dla_status check_shape(int dk, int dv) {
  if (dk != dv) return fail(DLA_ERR_UNSUPPORTED, "d_k (%d) != d_v (%d) is not built", dk, dv);
  if (dk != 64 && dk != 128) return fail(DLA_ERR_UNSUPPORTED, "d = %d not built (64 or 128)", dk);
  return DLA_OK;
}

dla_status check_cache(const dla_cache* c, int B, int H, int C, int d) {
  if (!c->states || !c->slot || !c->n || !c->ibar || !c->m) return fail(DLA_ERR_INVALID_ARG, "cache has a NULL member");
  if (c->B != B || c->H != H || c->C != C || c->dk != d || c->dv != d)
    return fail(DLA_ERR_INVALID_ARG, "cache dims (B=%d H=%d C=%d dk=%d dv=%d) do not match the call (B=%d H=%d C=%d d=%d)",
                c->B, c->H, c->C, c->dk, c->dv, B, H, C, d);
  if (!aligned(c->states, 16) || !aligned(c->ibar, 8) || !aligned(c->slot, 4) || !aligned(c->n, 4) || !aligned(c->m, 4))
    return fail(DLA_ERR_INVALID_ARG, "cache arrays are misaligned (states need 16 bytes)");
  return DLA_OK;
}

dla_status cuda_fail(cudaError_t e, const char* what) {
  return fail(DLA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// ---- internal streams of the overlapped forward schedule, one set per host
// thread and device: the scan runs on a high-priority stream, the read-out on
// a low-priority one, so the scan's few CTAs get SMs first.
struct StreamSet {
  cudaStream_t hi = nullptr, lo = nullptr;  // scan, read-out
  cudaStream_t cp = nullptr;                // host-to-device copies of streamed inputs
  cudaStream_t cpo = nullptr;               // device-to-host copies of the streamed output
  cudaEvent_t in = nullptr, gram_done = nullptr, scan_done[2] = {nullptr, nullptr}, ro_done[2] = {nullptr, nullptr};
  cudaEvent_t prep_done = nullptr, cp_done = nullptr, cpo_done = nullptr;
  bool ready = false;
};
constexpr int kMaxDev = 64;
thread_local StreamSet g_sets[kMaxDev];

cudaError_t stream_set(StreamSet** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
  StreamSet& S = g_sets[dev];
  if (!S.ready) {
    int least = 0, greatest = 0;
    if ((e = cudaDeviceGetStreamPriorityRange(&least, &greatest)) != cudaSuccess) return e;
    if ((e = cudaStreamCreateWithPriority(&S.hi, cudaStreamNonBlocking, greatest)) != cudaSuccess) return e;
    if ((e = cudaStreamCreateWithPriority(&S.lo, cudaStreamNonBlocking, least)) != cudaSuccess) return e;
    if ((e = cudaStreamCreateWithFlags(&S.cp, cudaStreamNonBlocking)) != cudaSuccess) return e;
    if ((e = cudaStreamCreateWithFlags(&S.cpo, cudaStreamNonBlocking)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&S.cp_done, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&S.cpo_done, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&S.in, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&S.gram_done, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&S.prep_done, cudaEventDisableTiming)) != cudaSuccess) return e;
    for (int i = 0; i < 2; ++i) {
      if ((e = cudaEventCreateWithFlags(&S.scan_done[i], cudaEventDisableTiming)) != cudaSuccess) return e;
      if ((e = cudaEventCreateWithFlags(&S.ro_done[i], cudaEventDisableTiming)) != cudaSuccess) return e;
    }
    S.ready = true;
  }
  *out = &S;
  return cudaSuccess;
}

// ---- device status of each stream (dla_sync_status)
// One word per (device, stream) in a static device array of the library
// (nothing is allocated): every call folds its device status into its
// stream's word (the first failure sticks) and dla_sync_status reads and
// clears it.  Streams are given words in the order they are first used; past
// kStatusWords - 1 streams on a device, the rest share the last word.
constexpr int kStatusWords = 256;
static __device__ int32_t g_status_board[kStatusWords];

struct StatusBoard {
  std::mutex mu;
  int32_t* base = nullptr;  // device address of g_status_board on this device
  std::vector<std::pair<cudaStream_t, int>> words;
};
StatusBoard g_board[64];

// The first failure of a call (its workspace status word) into its stream's word.
__global__ void status_fold_kernel(const int32_t* call_status, int32_t* word) {
  const int v = *(volatile const int32_t*)call_status;
  if (v != 0) atomicCAS(word, 0, v);
}

// Device address of the status word of `s` on the current device.
cudaError_t status_word(cudaStream_t s, int32_t** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  StatusBoard& B = g_board[dev];
  std::lock_guard<std::mutex> g(B.mu);
  if (!B.base) {
    // the module holding the board and the fold kernel is loaded here, before
    // any kernel of the call that might wait on another is enqueued
    cudaFuncAttributes fa;
    if ((e = cudaFuncGetAttributes(&fa, status_fold_kernel)) != cudaSuccess) return e;
    void* a = nullptr;
    if ((e = cudaGetSymbolAddress(&a, g_status_board)) != cudaSuccess) return e;
    B.base = (int32_t*)a;
  }
  int w = -1;
  for (const auto& p : B.words)
    if (p.first == s) w = p.second;
  if (w < 0) {
    w = (int)B.words.size() < kStatusWords - 1 ? (int)B.words.size() : kStatusWords - 1;
    B.words.emplace_back(s, w);
  }
  *out = B.base + w;
  return cudaSuccess;
}

// Debugging knobs of the failure-detection tests (environment variables read at
// every call; unset in normal use):
//   DLA_DEBUG_WAIT_MS=x       bounded device waits give up after about x ms
//                             instead of about 2 s;
//   DLA_DEBUG_WITHHOLD_PIECES=1  dla_forward_host copies every input piece but
//                             reports only the first as arrived, so a scan
//                             waiting for a later piece gives up (status 5).
int debug_wait_units() {  // the wait limit in units of 1024 SM clocks (0: default)
  const char* v = getenv("DLA_DEBUG_WAIT_MS");
  if (!v) return 0;
  const double ms = atof(v);
  if (!(ms > 0.0)) return 0;
  const double units = ms * 2.07e6 / 1024.0;  // SM clocks at 2.07 GHz
  return units < 1.0 ? 1 : (units > 2e9 ? 2000000000 : (int)units);
}
bool debug_withhold_pieces() {
  const char* v = getenv("DLA_DEBUG_WITHHOLD_PIECES");
  return v && strcmp(v, "1") == 0;
}

// ---- inputs in host memory (dla_forward_host)
// A 32-bit write to device memory in stream order, after the stream's earlier
// work and with a memory barrier before it (the driver's stream memory
// operation: no kernel, so it needs no SM while kernels wait for it).
typedef CUresult (*WriteValue32Fn)(CUstream, CUdeviceptr, cuuint32_t, unsigned int);
WriteValue32Fn write_value_fn() {
  static WriteValue32Fn fn = nullptr;
  static bool tried = false;
  static std::mutex mu;
  std::lock_guard<std::mutex> g(mu);
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuStreamWriteValue32", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<WriteValue32Fn>(p);
  }
  return fn;
}

// A stream wait until a 32-bit word of device memory is >= a value (the
// driver's stream memory operation: the stream, not an SM, waits).
typedef CUresult (*WaitValue32Fn)(CUstream, CUdeviceptr, cuuint32_t, unsigned int);
WaitValue32Fn wait_value_fn() {
  static WaitValue32Fn fn = nullptr;
  static bool tried = false;
  static std::mutex mu;
  std::lock_guard<std::mutex> g(mu);
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuStreamWaitValue32", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<WaitValue32Fn>(p);
  }
  return fn;
}

// q, k, v, lambda in host memory and their device copies in the workspace;
// o in host memory (copied back by the forward pass when it streams, else by
// the caller).
struct HostIO {
  const void* qh;
  const void* kh;
  const void* vh;
  const float* lamh;
  void* qd;
  void* kd;
  void* vd;
  float* lamd;
  size_t elt;  // bytes per q, k, v element
  void* oh;    // host output, or nullptr
  size_t oelt; // bytes per o element
  bool o_streamed = false;  // set by the forward pass: o was copied back piece by piece
};
// Tokens [t0, t1) of every batch row of k, v, q and lambda to the device, on stream s.
cudaError_t h2d_tokens(const HostIO& io, int B, int T, int H, int d, int C, int t0, int t1, cudaStream_t s) {
  cudaError_t e = cudaSuccess;
  for (int b = 0; b < B && e == cudaSuccess; ++b) {
    const size_t off = ((size_t)b * T + t0) * H * d * io.elt, n = (size_t)(t1 - t0) * H * d * io.elt;
    const void* src[3] = {io.kh, io.vh, io.qh};
    void* dst[3] = {io.kd, io.vd, io.qd};
    for (int i = 0; i < 3 && e == cudaSuccess; ++i)
      if (src[i]) e = cudaMemcpyAsync((char*)dst[i] + off, (const char*)src[i] + off, n, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess && io.lamh) {
      const size_t lo = ((size_t)b * T + t0) * H * C, ln = (size_t)(t1 - t0) * H * C;
      e = cudaMemcpyAsync(io.lamd + lo, io.lamh + lo, ln * sizeof(float), cudaMemcpyHostToDevice, s);
    }
  }
  return e;
}

// ---- optional per-launch CUDA-event timing (dla_timing_enable / _read)
struct TimedLaunch {
  int kind;
  cudaEvent_t start, stop;
};
thread_local bool g_timing = false;
thread_local std::vector<TimedLaunch> g_records;
thread_local std::vector<cudaEvent_t> g_free_events;

cudaEvent_t take_event() {
  if (!g_free_events.empty()) {
    cudaEvent_t e = g_free_events.back();
    g_free_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Runs one launch, bracketed by events when timing is enabled.
template <typename F>
cudaError_t timed(int kind, cudaStream_t st, F&& launch) {
  if (!g_timing) return launch();
  TimedLaunch r{kind, take_event(), take_event()};
  if (!r.start || !r.stop) return cudaErrorMemoryAllocation;
  cudaEventRecord(r.start, st);
  cudaError_t e = launch();
  cudaEventRecord(r.stop, st);
  g_records.push_back(r);
  return e;
}

}  // namespace

namespace dla {
dla_status set_error(dla_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}
}  // namespace dla

extern "C" {

void dla_default_params(dla_params* p) {
  if (!p) return;
  p->tau = 0.6;
  p->eps = 1e-6;
  p->rms_eps = 1e-6;
  p->capacity = 30;
  p->score_mode = 0;
  p->out_dtype = DLA_F32;
  p->from_cache = 0;
  p->seq_lens = nullptr;
}

int dla_version(void) { return DLA_VERSION; }

dla_status dla_timing_enable(int enable) {
  g_timing = (enable != 0);
  return ok();
}

dla_status dla_timing_read(int* launches, double* ms, int reset) {
  if (!launches || !ms) return fail(DLA_ERR_INVALID_ARG, "launches and ms must be non-NULL");
  for (int k = 0; k < DLA_K_COUNT; ++k) {
    launches[k] = 0;
    ms[k] = 0.0;
  }
  for (const TimedLaunch& r : g_records) {
    cudaError_t e = cudaEventSynchronize(r.stop);
    if (e != cudaSuccess) return cuda_fail(e, "timing event");
    float t = 0.f;
    e = cudaEventElapsedTime(&t, r.start, r.stop);
    if (e != cudaSuccess) return cuda_fail(e, "timing elapsed");
    launches[r.kind] += 1;
    ms[r.kind] += t;
  }
  if (reset) {
    for (const TimedLaunch& r : g_records) {
      g_free_events.push_back(r.start);
      g_free_events.push_back(r.stop);
    }
    g_records.clear();
  }
  return ok();
}

dla_status dla_sync_status(void* stream) {
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  int32_t* word = nullptr;
  if ((e = status_word(s, &word)) != cudaSuccess) return cuda_fail(e, "status word");
  int32_t v = 0;
  if ((e = cudaMemcpyAsync(&v, word, sizeof(v), cudaMemcpyDeviceToHost, s)) != cudaSuccess ||
      (e = cudaMemsetAsync(word, 0, sizeof(int32_t), s)) != cudaSuccess || (e = cudaStreamSynchronize(s)) != cudaSuccess)
    return cuda_fail(e, "status read");
  switch (v) {
    case 0: return ok();
    case DLA_ERR_TIMEOUT:
      return fail(DLA_ERR_TIMEOUT, "a bounded device wait gave up in a call on this stream (its outputs are undefined)");
    case DLA_ERR_DEVICE_CHECK:
      return fail(DLA_ERR_DEVICE_CHECK, "a device-side consistency check failed in a call on this stream");
    default:
      return fail(DLA_ERR_DEVICE_CHECK, "unexpected device status %d on this stream", v);
  }
}

const char* dla_last_error(void) { return g_err; }

const char* dla_status_string(dla_status s) {
  switch (s) {
    case DLA_OK: return "DLA_OK";
    case DLA_ERR_INVALID_ARG: return "DLA_ERR_INVALID_ARG";
    case DLA_ERR_UNSUPPORTED: return "DLA_ERR_UNSUPPORTED";
    case DLA_ERR_WORKSPACE: return "DLA_ERR_WORKSPACE";
    case DLA_ERR_CUDA: return "DLA_ERR_CUDA";
    case DLA_ERR_TIMEOUT: return "DLA_ERR_TIMEOUT";
    case DLA_ERR_DEVICE_CHECK: return "DLA_ERR_DEVICE_CHECK";
  }
  return "DLA_ERR_UNKNOWN";
}

size_t dla_cache_bytes(int B, int H, int C, int dk, int dv) {
  if (B < 1 || H < 1 || C < 1 || dk < 1 || dv < 1) return 0;
  return cache_layout(B, H, C, dk, dv).total;
}

dla_status dla_cache_carve(void* base, size_t bytes, int B, int H, int C, int dk, int dv, dla_cache* out) {
  if (!base || !out) return fail(DLA_ERR_INVALID_ARG, "base and out must be non-NULL");
  if (B < 1 || H < 1 || C < 2 || dk < 1 || dv < 1) return fail(DLA_ERR_INVALID_ARG, "bad cache dims");
  if (!aligned(base, 256)) return fail(DLA_ERR_INVALID_ARG, "cache base must be 256-byte aligned");
  CacheLayout L = cache_layout(B, H, C, dk, dv);
  if (bytes < L.total) return fail(DLA_ERR_WORKSPACE, "cache block has %zu bytes, needs %zu", bytes, L.total);
  char* c = (char*)base;
  out->states = (float*)(c + L.states);
  out->slot = (int32_t*)(c + L.slot);
  out->n = (int32_t*)(c + L.n);
  out->ibar = (double*)(c + L.ibar);
  out->m = (int32_t*)(c + L.m);
  out->B = B; out->H = H; out->C = C; out->dk = dk; out->dv = dv;
  return ok();
}

dla_status dla_init_cache(const dla_cache* cache, void* stream) {
  if (!cache) return fail(DLA_ERR_INVALID_ARG, "cache is NULL");
  if (cache->B < 1 || cache->H < 1 || cache->C < 2) return fail(DLA_ERR_INVALID_ARG, "bad cache dims");
  if (!cache->slot || !cache->n || !cache->ibar || !cache->m) return fail(DLA_ERR_INVALID_ARG, "cache has a NULL member");
  cudaError_t e = timed(DLA_K_INIT, (cudaStream_t)stream, [&] {
    return dla::launch_init_cache(cache->slot, cache->n, cache->ibar, cache->m, cache->B * cache->H, cache->C,
                                  (cudaStream_t)stream);
  });
  if (e != cudaSuccess) return cuda_fail(e, "init_cache launch");
  return ok();
}

static FwdPlan choose_plan(const dla_params* p, int B, int T, int H, int d, dla_dtype in_dtype, bool with_output,
                           bool need_trace, bool need_cache, size_t budget) {
  const int nsnap = (T + readout_interval(in_dtype, d) - 1) / readout_interval(in_dtype, d);
  if (!with_output) return plan_for(1, false, p, B, T, H, d, in_dtype, false, need_trace, need_cache);
  // about kTargetRounds rounds, so that all but the last read-out hide behind the scan
  const int rounds = nsnap < kTargetRounds ? nsnap : kTargetRounds;
  const int R = (nsnap + rounds - 1) / rounds;
  FwdPlan pp = plan_for(R, true, p, B, T, H, d, in_dtype, true, need_trace, need_cache);
  if (pp.total <= budget) return pp;
  auto reset = [&](int r) { return plan_for(r, false, p, B, T, H, d, in_dtype, true, need_trace, need_cache); };
  if (reset(R).total <= budget || reset(1).total > budget) return reset(reset(R).total <= budget ? R : 1);
  int lo = 1, hi = R;  // the largest round that fits
  while (lo < hi) {
    const int mid = lo + (hi - lo + 1) / 2;
    if (reset(mid).total <= budget) lo = mid;
    else hi = mid - 1;
  }
  return reset(lo);
}

size_t dla_forward_workspace(const dla_params* p, int B, int T, int H, int dk, int dv, dla_dtype in_dtype,
                             int with_output) {
  if (!p || B < 1 || T < 1 || H < 1 || dk < 1 || dv < 1) return 0;
  // sized for the worst case of the call: trace and cache held in the workspace
  return choose_plan(p, B, T, H, dk, in_dtype, with_output != 0, true, true, kPreferredWorkspace).total;
}

size_t dla_forward_min_workspace(const dla_params* p, int B, int T, int H, int dk, int dv, dla_dtype in_dtype,
                                 int with_output) {
  if (!p || B < 1 || T < 1 || H < 1 || dk < 1 || dv < 1) return 0;
  return plan_for(1, false, p, B, T, H, dk, in_dtype, with_output != 0, true, true).total;
}

// SMs the scan leaves to the rest on the concurrent schedule when all its CTAs
// are resident (0: they are not)
static int concurrent_free_sms(int B, int H, int d, bool scan_tc, cudaError_t* err) {
  int dev = 0, sms = 0;
  if ((*err = cudaGetDevice(&dev)) != cudaSuccess ||
      (*err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return 0;
  const int BH = B * H;
  if (scan_tc) return (dla::scan_tc_resident_streams() >= BH) ? sms - BH : 0;
  return (dla::scan_mma_resident_streams(BH, d) >= BH) ? sms - BH * dla::scan_mma_ctas_per_stream(BH, d) : 0;
}

// dla_forward; with io, q, k, v and lambda come from host memory into the
// device buffers q, k, v, lam (workspace), streamed beside the scan on the
// concurrent schedule, otherwise copied before anything else.
// A packed batch: row b holds tokens cu[b] .. cu[b+1] - 1 of q, k, v, lambda and o
// (device int32 offsets), `total` token rows in all.
struct Varlen {
  const int32_t* cu;
  long long total;
};

static dla_status forward_launch(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv,
                                 const void* q, const void* k, const void* v, const float* lam, void* o,
                                 const dla_cache* cache, uint8_t* boundary, int32_t* merge_log, void* workspace,
                                 size_t ws_bytes, void* stream, HostIO* io, const Varlen* vl, int32_t** word);

// forward_launch, then the call's device status folded into its stream's status
// word once every kernel of the call has run (the stream waits for them).
static dla_status forward_impl(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv,
                               const void* q, const void* k, const void* v, const float* lam, void* o,
                               const dla_cache* cache, uint8_t* boundary, int32_t* merge_log, void* workspace,
                               size_t ws_bytes, void* stream, HostIO* io, const Varlen* vl = nullptr) {
  int32_t* word = nullptr;
  dla_status s = forward_launch(p, in_dtype, B, T, H, dk, dv, q, k, v, lam, o, cache, boundary, merge_log, workspace,
                                ws_bytes, stream, io, vl, &word);
  if (s != DLA_OK) return s;
  cudaError_t e = timed(DLA_K_STATUS, (cudaStream_t)stream, [&] {
    status_fold_kernel<<<1, 1, 0, (cudaStream_t)stream>>>((const int32_t*)workspace, word);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return cuda_fail(e, "status fold launch");
  return ok();
}

static dla_status forward_launch(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv,
                                 const void* q, const void* k, const void* v, const float* lam, void* o,
                                 const dla_cache* cache, uint8_t* boundary, int32_t* merge_log, void* workspace,
                                 size_t ws_bytes, void* stream, HostIO* io, const Varlen* vl, int32_t** word) {
  dla_status s = check_params(p);
  if (s != DLA_OK) return s;
  if (in_dtype != DLA_BF16 && in_dtype != DLA_F32) return fail(DLA_ERR_INVALID_ARG, "bad in_dtype");
  if (B < 1 || T < 1 || H < 1) return fail(DLA_ERR_INVALID_ARG, "B, T, H must be >= 1");
  if ((s = check_shape(dk, dv)) != DLA_OK) return s;
  const int d = dk, C = p->capacity;
  if ((long long)B * T * H * d >= (1LL << 40)) return fail(DLA_ERR_UNSUPPORTED, "tensor too large");
  if (C > dla::kMaxC) {  // the DLA(I) instances (no capacity merge)
    if (in_dtype != DLA_BF16 || d != 128)
      return fail(DLA_ERR_UNSUPPORTED, "capacity %d > %d needs bf16 inputs with d = 128", C, dla::kMaxC);
    if (p->seq_lens || vl || io)
      return fail(DLA_ERR_UNSUPPORTED, "capacity %d > %d takes whole rows of device-resident inputs", C, dla::kMaxC);
  }
  if (vl) {
    if (!vl->cu || !aligned(vl->cu, 4)) return fail(DLA_ERR_INVALID_ARG, "cu_seqlens must be non-NULL and 4-byte aligned");
    if (p->seq_lens) return fail(DLA_ERR_INVALID_ARG, "a packed batch takes its lengths from cu_seqlens: seq_lens must be NULL");
    if (vl->total < 0 || vl->total >= (1LL << 31)) return fail(DLA_ERR_UNSUPPORTED, "total_tokens must be in [0, 2^31)");
    if (vl->total * H * d >= (1LL << 40)) return fail(DLA_ERR_UNSUPPORTED, "tensor too large");
    if (io) return fail(DLA_ERR_UNSUPPORTED, "packed batches take device-resident inputs");
  }
  // the host copies move whole rows, so the o rows past a row's length could not
  // stay unwritten, as seq_lens promises
  if (io && p->seq_lens) return fail(DLA_ERR_UNSUPPORTED, "per-row lengths (seq_lens) take device-resident inputs");
  if (!k || !v) return fail(DLA_ERR_INVALID_ARG, "k and v must be non-NULL");
  const bool with_output = (o != nullptr);
  if (with_output && !q) return fail(DLA_ERR_INVALID_ARG, "q must be non-NULL when o is requested");
  const size_t vec = 16;
  if (!aligned(k, vec) || !aligned(v, vec) || (q && !aligned(q, vec)) || (o && !aligned(o, vec)))
    return fail(DLA_ERR_INVALID_ARG, "q, k, v, o must be 16-byte aligned");
  if (lam && !aligned(lam, 4)) return fail(DLA_ERR_INVALID_ARG, "lambda must be 4-byte aligned");
  if (p->seq_lens && !aligned(p->seq_lens, 4)) return fail(DLA_ERR_INVALID_ARG, "seq_lens must be 4-byte aligned");
  if (cache) {
    if ((s = check_cache(cache, B, H, C, d)) != DLA_OK) return s;
  } else if (p->from_cache) {
    return fail(DLA_ERR_INVALID_ARG, "from_cache = 1 needs a cache");
  }
  if (!workspace) return fail(DLA_ERR_WORKSPACE, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(DLA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const bool need_trace = (boundary == nullptr) || (merge_log == nullptr);
  const bool need_cache = (cache == nullptr);
  FwdPlan P = choose_plan(p, B, T, H, d, in_dtype, with_output, need_trace, need_cache, ws_bytes);
  if (P.total > ws_bytes)
    return fail(DLA_ERR_WORKSPACE, "workspace has %zu bytes, needs at least %zu", ws_bytes, P.total);

  cudaStream_t st = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  int32_t* status = (int32_t*)(ws + P.off_status);
  bool stream_in = false;  // inputs from host memory streamed beside the scan
  if (io) {
    cudaError_t qe = cudaSuccess;
    stream_in = with_output && use_tc(in_dtype, d) && P.persistent && (P.nsnap_total + 1) / 2 <= 65535 &&
                schedule() == kConcurrent && concurrent_free_sms(B, H, d, false, &qe) >= kMinFreeSms && write_value_fn();
    if (qe != cudaSuccess) return cuda_fail(qe, "device query");
    if (!stream_in) {
      const cudaError_t ce = h2d_tokens(*io, B, T, H, d, C, 0, T, st);
      if (ce != cudaSuccess) return cuda_fail(ce, "input copy");
    }
  }
  uint8_t* bnd = boundary ? boundary : (uint8_t*)(ws + P.off_bnd);
  int32_t* mlog = merge_log ? merge_log : (int32_t*)(ws + P.off_mlog);
  dla_cache live;
  if (cache) {
    live = *cache;
  } else {
    dla_cache_carve(ws + P.off_cache, cache_layout(B, H, C, d, d).total, B, H, C, d, d, &live);
  }
  // the stream's status word (looked up before anything is enqueued), the call's
  // status word and, after it, the wait limit of its kernels (0: default)
  cudaError_t e = status_word(st, word);
  if (e != cudaSuccess) return cuda_fail(e, "status word");
  e = cudaMemsetAsync(status, 0, 2 * sizeof(int32_t), st);
  if (e != cudaSuccess) return cuda_fail(e, "status reset");
  if (const int wu = debug_wait_units()) {
    if (!write_value_fn() ||
        write_value_fn()((CUstream)st, (CUdeviceptr)(status + 1), (cuuint32_t)wu, 0) != CUDA_SUCCESS)
      return fail(DLA_ERR_CUDA, "stream memory write of the debug wait limit failed");
  }
  if (!p->from_cache) {
    e = timed(DLA_K_INIT, st, [&] { return dla::launch_init_cache(live.slot, live.n, live.ibar, live.m, B * H, C, st); });
    if (e != cudaSuccess) return cuda_fail(e, "init_cache launch");
  }
  // per-row lengths (ragged rows in the padded layout, or a packed batch's rows,
  // checked on the device) and, for a packed batch, each row's first token row
  const int32_t* seq_lens = p->seq_lens;
  const int32_t* row_start = nullptr;
  if (vl) {
    int32_t* lens_ws = (int32_t*)(ws + P.off_rows);
    int32_t* start_ws = lens_ws + B;
    e = timed(DLA_K_INIT, st, [&] { return dla::launch_varlen_rows(vl->cu, B, T, vl->total, lens_ws, start_ws, status, st); });
    if (e != cudaSuccess) return cuda_fail(e, "packed rows launch");
    seq_lens = lens_ws;
    row_start = start_ws;
  }

  dla::ScanArgs sa;
  memset(&sa, 0, sizeof(sa));
  sa.k = k; sa.v = v;
  sa.B = B; sa.T = T; sa.H = H;
  sa.sp.tau = p->tau; sa.sp.eps = p->eps; sa.sp.rms_eps = p->rms_eps; sa.sp.score_mode = p->score_mode;
  dla::finish_score_params(sa.sp);
  sa.C = C;
  sa.states = live.states; sa.slot = live.slot; sa.n = live.n; sa.ibar = live.ibar; sa.m = live.m;
  sa.boundary = bnd; sa.merge_log = mlog;
  sa.status = status;
  sa.seq_lens = seq_lens;
  sa.row_start = row_start;
  const bool in_bf16 = (in_dtype == DLA_BF16);
  const bool tc = use_tc(in_dtype, d);
  const bool pool_f16 = tc;  // fp16 pool entries for the tensor-core read-out, else fp32
  if (!with_output) {
    sa.t_begin = 0; sa.t_end = T;
    sa.pool = nullptr; sa.pool_cap = 0; sa.nsnap = 1; sa.snap_chunks = 1;
    e = timed(DLA_K_SCAN, st, [&] { return (in_bf16 ? dla::launch_scan_mma(sa, d, pool_f16, st) : dla::launch_scan(sa, d, st)); });
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    return ok();
  }
  dla::ReadoutArgs ra;
  memset(&ra, 0, sizeof(ra));
  ra.q = q; ra.k = k; ra.v = v; ra.lam = lam; ra.o = o;
  ra.out_bf16 = (p->out_dtype == DLA_BF16);
  ra.B = B; ra.T = T; ra.H = H; ra.C = C;
  ra.boundary = bnd; ra.merge_log = mlog;
  ra.status = status;
  ra.seq_lens = seq_lens;
  ra.row_start = row_start;
  ra.total_rows = vl ? vl->total : 0;
  ra.interval = P.interval;
  sa.snap_chunks = P.interval / dla::kScanL;
  sa.pool_cap = P.pool_cap;
  ra.pool_cap = P.pool_cap;
  sa.snap_stride = ra.snap_stride = P.nsnap_total;
  sa.snap_m0 = (int32_t*)(ws + P.off_lists_m0);
  sa.snap_ids = (int32_t*)(ws + P.off_lists_ids);
  ra.snap_m0 = sa.snap_m0;
  ra.snap_ids = sa.snap_ids;
  sa.pstate = P.persistent ? (int32_t*)(ws + P.off_pstate) : nullptr;
  sa.nbound = (float*)(ws + P.off_nbound);
  if (tc && p->from_cache) {  // the continued cache's norm bounds, for the scales of its snapshots
    e = timed(DLA_K_INIT, st, [&] {
      return dla::launch_cache_bounds(live.states, live.slot, live.m, B * H, C, d, sa.nbound, st);
    });
    if (e != cudaSuccess) return cuda_fail(e, "cache bounds launch");
  }
  sa.gram = P.gram_chunks ? (const float*)(ws + P.off_gram) : nullptr;
  sa.gram_chunks = P.gram_chunks;
  // The scan: the mma.sync scan (CTA pairs, the open state in registers) by
  // default; with DLA_SCAN=tc, on tcgen05 with the open state in tensor memory
  // (one CTA per stream) where the Gram pre-pass runs over whole rows of
  // resident inputs (it is correct but slower on the benchmark workloads:
  // its per-chunk chain is bound by the latency of small tensor-core groups).
  const bool scan_tc = tc && C <= dla::kMaxC && P.gram_chunks > 0 && !seq_lens && !stream_in && scan_tc_requested();
  auto launch_main_scan = [&](cudaStream_t s_) -> cudaError_t {
    return scan_tc ? dla::launch_scan_tc(sa, s_) : dla::launch_scan_mma(sa, d, pool_f16, s_);
  };
  const int gram_per_sm = scan_tc ? dla::kGramTcCtasPerSm : dla::kGramCtasPerSm;
  // Round r: the scan (high-priority stream) appends to the pool, then the
  // read-out of round r (low-priority stream) runs while the scan of round
  // r + 1 proceeds.  In reset mode pool b is reused by round r + 2 only after
  // the read-out of round r has finished.
  StreamSet* S = nullptr;
  if ((e = stream_set(&S)) != cudaSuccess) return cuda_fail(e, "internal streams");
  if ((e = cudaEventRecord(S->in, st)) != cudaSuccess) return cuda_fail(e, "event record");
  if ((e = cudaStreamWaitEvent(S->hi, S->in, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  const Schedule sched = schedule();
  const bool one_readout = P.persistent && tc && (P.nsnap_total + 1) / 2 <= 65535;  // one read-out launch
  if (one_readout && sched == kSerial) {
    // pre-pass, whole scan, read-out, one after another on the scan stream
    dla::GramArgs ga;
    ga.k = k; ga.v = v; ga.B = B; ga.T = T; ga.H = H; ga.nchunks = P.gram_chunks;
    ga.seq_lens = seq_lens; ga.row_start = row_start;
    ga.out = (float*)(ws + P.off_gram);
    ga.chunk0 = 0; ga.count = P.gram_chunks;
    ga.ready = nullptr;
    ga.packed = scan_tc ? 1 : 0;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess || (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e, "device query");
    dla::gram_blocks(B * H, P.gram_chunks, gram_per_sm * sms, &ga.nblk, &ga.per_blk);
    if (P.gram_chunks) {
      e = timed(DLA_K_GRAM, S->hi, [&] { return dla::launch_gram(ga, d, S->hi); });
      if (e != cudaSuccess) return cuda_fail(e, "gram launch");
    }
    sa.pool = ws + P.off_pool;
    sa.pool_scale = (float*)((char*)sa.pool + P.pool_scale_off);
    sa.t_begin = 0; sa.t_end = T;
    sa.nsnap = P.nsnap_total; sa.snap_base = 0;
    sa.carry_in = 0; sa.snap_at_end = 0;
    e = timed(DLA_K_SCAN, S->hi, [&] { return launch_main_scan(S->hi); });
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    ra.pool = sa.pool;
    ra.pool_scale = sa.pool_scale;
    ra.t_begin = 0; ra.t_end = T;
    ra.nsnap = P.nsnap_total; ra.snap_base = 0;
    e = timed(DLA_K_READOUT, S->hi, [&] { return dla::launch_readout_tc(ra, status, S->hi); });
    if (e != cudaSuccess) return cuda_fail(e, "readout launch");
    if ((e = cudaEventRecord(S->scan_done[0], S->hi)) != cudaSuccess) return cuda_fail(e, "event record");
    if ((e = cudaStreamWaitEvent(st, S->scan_done[0], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    return ok();
  }
  int free_sms = 0;  // SMs the scan leaves to the rest when all its CTAs are resident (0: they are not)
  if (one_readout && sched == kConcurrent) {
    free_sms = concurrent_free_sms(B, H, d, scan_tc, &e);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
  }
  if (free_sms >= kMinFreeSms) {
    // One scan over the whole sequence (high-priority stream) and the read-out
    // in rounds beside it (low-priority streams): each read-out CTA waits for its
    // stream's progress, so rounds never wait for the slowest stream and the
    // scan is launched once.  A one-CTA gate holds the other streams until
    // every scan CTA has started, so that nothing launched beside the scan
    // takes an SM the scan needs.  Then the Gram pre-pass runs on the free SMs
    // while the scan consumes it chunk by chunk (per-block counters), and the
    // read-out follows the pre-pass (a waiting read-out CTA must not hold an SM
    // the pre-pass needs).  Needs every scan CTA resident at once, with SMs to
    // spare; otherwise the rounds schedule below runs.
    {  // kernel code loaded once per device before anything of this path runs
      static bool loaded[kMaxDev] = {};
      static std::mutex mu;
      int dev = 0;
      if ((e = cudaGetDevice(&dev)) != cudaSuccess || dev < 0 || dev >= kMaxDev) return cuda_fail(e, "device query");
      std::lock_guard<std::mutex> g(mu);
      if (!loaded[dev]) {
        if ((e = dla::preload_scan_kernels()) != cudaSuccess || (e = dla::preload_scan_tc_kernel()) != cudaSuccess ||
            (e = dla::preload_readout_kernels()) != cudaSuccess)
          return cuda_fail(e, "kernel load");
        loaded[dev] = true;
      }
    }
    int32_t* progress = (int32_t*)(ws + P.off_progress);
    int32_t* started = progress + 2 * B * H;
    int32_t* pieces = started + 1;  // input pieces streamed in so far
    int32_t* out_done = started + 2;  // [kOutPieces] read-out CTAs done per output piece
    int32_t* gram_ready = out_done + kOutPieces;
    // with streamed inputs the scan forms its Gram entries itself: a pre-pass
    // waiting for the pieces would hold back the read-out behind it
    const bool run_gram = P.gram_chunks && !stream_in;
    const int ctas = scan_tc ? 1 : dla::scan_mma_ctas_per_stream(B * H, d);
    dla::GramArgs ga;
    ga.k = k; ga.v = v; ga.B = B; ga.T = T; ga.H = H; ga.nchunks = P.gram_chunks;
    ga.seq_lens = seq_lens; ga.row_start = row_start;
    ga.out = (float*)(ws + P.off_gram);
    ga.chunk0 = 0; ga.count = P.gram_chunks;
    ga.ready = gram_ready;
    ga.packed = scan_tc ? 1 : 0;
    dla::gram_blocks(B * H, P.gram_chunks, gram_per_sm * free_sms, &ga.nblk, &ga.per_blk);
    if ((e = cudaMemsetAsync(progress, 0, (2 * B * H + 2 + kOutPieces + B * H * ga.nblk) * sizeof(int32_t), S->hi)) !=
        cudaSuccess)
      return cuda_fail(e, "progress reset");
    if ((e = cudaEventRecord(S->prep_done, S->hi)) != cudaSuccess) return cuda_fail(e, "event record");
    if ((e = cudaStreamWaitEvent(S->lo, S->prep_done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    sa.pool = ws + P.off_pool;
    sa.pool_scale = (float*)((char*)sa.pool + P.pool_scale_off);
    sa.t_begin = 0; sa.t_end = T;
    sa.nsnap = P.nsnap_total; sa.snap_base = 0;
    sa.carry_in = 0; sa.snap_at_end = 0;
    sa.progress = progress; sa.started = started;
    if (run_gram) {
      sa.gram_ready = gram_ready;
      sa.gram_nblk = ga.nblk;
    } else {
      sa.gram = nullptr;
    }
    // Streamed inputs: pieces of pc chunks on the copy stream, each followed by
    // the count of pieces in place (a stream memory write); the scan waits for
    // the piece of each chunk it loads, the read-out for the scan.
    int pc = 0, npiece = 0;
    const bool withhold = stream_in && debug_withhold_pieces();
    auto put_piece = [&](int pi) -> dla_status {
      const int t0 = pi * pc * dla::kScanL, t1 = std::min(T, (pi + 1) * pc * dla::kScanL);
      const cudaError_t ce = h2d_tokens(*io, B, T, H, d, C, t0, t1, S->cp);
      if (ce != cudaSuccess) return cuda_fail(ce, "input copy");
      if (pi > 0 && withhold) return DLA_OK;  // debugging: later pieces never reported
      if (write_value_fn()((CUstream)S->cp, (CUdeviceptr)pieces, (cuuint32_t)(pi + 1), 0) != CUDA_SUCCESS)
        return fail(DLA_ERR_CUDA, "stream memory write failed");
      return DLA_OK;
    };
    if (stream_in) {
      const int nch = (T + dla::kScanL - 1) / dla::kScanL;
      pc = std::max(1, (nch + kInputPieces - 1) / kInputPieces);
      npiece = (nch + pc - 1) / pc;
      sa.piece_ready = pieces;
      sa.piece_chunks = pc;
      if ((e = cudaStreamWaitEvent(S->cp, S->prep_done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
      if ((s = put_piece(0)) != DLA_OK) return s;
    }
    e = timed(DLA_K_SCAN, S->hi, [&] { return launch_main_scan(S->hi); });
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    e = timed(DLA_K_GATE, S->lo, [&] { return dla::launch_gate(started, B * H * ctas, status, S->lo); });
    if (e != cudaSuccess) return cuda_fail(e, "gate launch");
    if (run_gram) {  // K0 beside the scan, on the SMs it leaves free
      e = timed(DLA_K_GRAM, S->lo, [&] { return dla::launch_gram(ga, d, S->lo); });
      if (e != cudaSuccess) return cuda_fail(e, "gram launch");
    }
    ra.pool = sa.pool;
    ra.pool_scale = sa.pool_scale;
    ra.progress = progress; ra.progress_ctas = ctas; ra.status = status;
    // the read-out follows the pre-pass on the read-out stream: one launch over
    // the whole sequence, its CTAs dispatched interval by interval (streams
    // fastest), each waiting for its stream's progress
    ra.t_begin = 0; ra.t_end = T;
    ra.nsnap = P.nsnap_total; ra.snap_base = 0;
    // Streamed output: pieces of opp interval pairs, each copied back once its
    // read-out CTAs are done (a stream wait on their count: the copy stream
    // waits, no SM does)
    const bool stream_out = stream_in && io->oh && wait_value_fn();
    const int npairs = (P.nsnap_total + 1) / 2;
    const int opp = std::max(1, (npairs + kOutPieces - 1) / kOutPieces), nop = (npairs + opp - 1) / opp;
    if (stream_out) {
      ra.out_done = out_done;
      ra.out_piece_pairs = opp;
    }
    ra.lam_l2 = stream_in ? 1 : 0;
    e = timed(DLA_K_READOUT, S->lo, [&] { return dla::launch_readout_tc(ra, status, S->lo); });
    if (e != cudaSuccess) return cuda_fail(e, "readout launch");
    if (stream_out) {
      if ((e = cudaStreamWaitEvent(S->cpo, S->prep_done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
      const int tp = 2 * P.interval;  // tokens per interval pair
      for (int op = 0; op < nop; ++op) {
        const int p0 = op * opp, p1 = std::min(npairs, p0 + opp);
        // one read-out CTA per (interval, stream): the piece's intervals
        const int nint = std::min(P.nsnap_total, 2 * p1) - 2 * p0;
        if (wait_value_fn()((CUstream)S->cpo, (CUdeviceptr)(out_done + op), (cuuint32_t)(B * H * nint), 0) !=
            CUDA_SUCCESS)
          return fail(DLA_ERR_CUDA, "stream memory wait failed");
        const int t0 = p0 * tp, t1 = std::min(T, p1 * tp);
        for (int b = 0; b < B; ++b) {
          const size_t off = ((size_t)b * T + t0) * H * d * io->oelt, n = (size_t)(t1 - t0) * H * d * io->oelt;
          if ((e = cudaMemcpyAsync((char*)io->oh + off, (const char*)o + off, n, cudaMemcpyDeviceToHost, S->cpo)) !=
              cudaSuccess)
            return cuda_fail(e, "output copy");
        }
      }
      if ((e = cudaEventRecord(S->cpo_done, S->cpo)) != cudaSuccess) return cuda_fail(e, "event record");
      if ((e = cudaStreamWaitEvent(st, S->cpo_done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
      io->o_streamed = true;
    }
    if (stream_in) {
      for (int pi = 1; pi < npiece; ++pi)
        if ((s = put_piece(pi)) != DLA_OK) return s;
      if ((e = cudaEventRecord(S->cp_done, S->cp)) != cudaSuccess) return cuda_fail(e, "event record");
      if ((e = cudaStreamWaitEvent(st, S->cp_done, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    }
    if ((e = cudaEventRecord(S->scan_done[0], S->hi)) != cudaSuccess) return cuda_fail(e, "event record");
    if ((e = cudaEventRecord(S->ro_done[0], S->lo)) != cudaSuccess) return cuda_fail(e, "event record");
    if ((e = cudaStreamWaitEvent(st, S->scan_done[0], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    if ((e = cudaStreamWaitEvent(st, S->ro_done[0], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    return ok();
  }
  const std::vector<int> sizes = round_sizes(P, P.persistent != 0);
  bool gram_rest = false;  // the scan of round 1 waits for the Gram tables of rounds 1..
  if (P.gram_chunks) {
    // K0: Gram suffix tables.  Round 0's chunks run ahead of the first scan on
    // the scan stream; the rest run on the read-out stream while that scan goes.
    dla::GramArgs ga;
    ga.k = k; ga.v = v; ga.B = B; ga.T = T; ga.H = H; ga.nchunks = P.gram_chunks;
    ga.seq_lens = seq_lens; ga.row_start = row_start;
    ga.out = (float*)(ws + P.off_gram);
    ga.ready = nullptr;
    ga.packed = scan_tc ? 1 : 0;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess || (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e, "device query");
    const int first = std::min(P.gram_chunks, sizes[0] * P.interval / dla::kScanL);
    ga.chunk0 = 0; ga.count = first;
    dla::gram_blocks(B * H, ga.count, gram_per_sm * sms, &ga.nblk, &ga.per_blk);
    e = timed(DLA_K_GRAM, S->hi, [&] { return dla::launch_gram(ga, d, S->hi); });
    if (e != cudaSuccess) return cuda_fail(e, "gram launch");
    if (first < P.gram_chunks) {
      ga.chunk0 = first; ga.count = P.gram_chunks - first;
      dla::gram_blocks(B * H, ga.count, gram_per_sm * sms, &ga.nblk, &ga.per_blk);
      if ((e = cudaStreamWaitEvent(S->lo, S->in, 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
      e = timed(DLA_K_GRAM, S->lo, [&] { return dla::launch_gram(ga, d, S->lo); });
      if (e != cudaSuccess) return cuda_fail(e, "gram launch");
      if ((e = cudaEventRecord(S->gram_done, S->lo)) != cudaSuccess) return cuda_fail(e, "event record");
      gram_rest = true;
    }
  }
  bool used[2] = {false, false};
  int snap0 = 0;  // global index of the round's first interval
  for (int r = 0; r < (int)sizes.size(); snap0 += sizes[r], ++r) {
    const int t0 = snap0 * P.interval;
    const int t1 = std::min(T, t0 + sizes[r] * P.interval);
    const int bsel = P.persistent ? 0 : (r % 2) % P.nbuf;
    sa.pool = ws + P.off_pool + (size_t)bsel * P.pool_bytes;
    sa.pool_scale = (float*)((char*)sa.pool + P.pool_scale_off);
    ra.pool = sa.pool;
    ra.pool_scale = sa.pool_scale;
    sa.t_begin = t0; sa.t_end = t1;
    sa.nsnap = (t1 - t0 + P.interval - 1) / P.interval;
    sa.snap_base = ra.snap_base = snap0;
    sa.carry_in = (P.persistent && r > 0) ? 1 : 0;
    sa.snap_at_end = (P.persistent && t1 < T) ? 1 : 0;
    if (!P.persistent && used[bsel] && (e = cudaStreamWaitEvent(S->hi, S->ro_done[bsel], 0)) != cudaSuccess)
      return cuda_fail(e, "stream wait");
    if (r == 1 && gram_rest && (e = cudaStreamWaitEvent(S->hi, S->gram_done, 0)) != cudaSuccess)
      return cuda_fail(e, "stream wait");
    e = timed(DLA_K_SCAN, S->hi, [&] {
      return in_bf16 ? launch_main_scan(S->hi) : dla::launch_scan(sa, d, S->hi);
    });
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    if ((e = cudaEventRecord(S->scan_done[r % 2], S->hi)) != cudaSuccess) return cuda_fail(e, "event record");
    if ((e = cudaStreamWaitEvent(S->lo, S->scan_done[r % 2], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
    ra.t_begin = t0; ra.t_end = t1; ra.nsnap = sa.nsnap;
    e = timed(DLA_K_READOUT, S->lo, [&] {
      return tc ? dla::launch_readout_tc(ra, status, S->lo)
                : dla::launch_readout_simt(ra, d, in_bf16, S->lo);
    });
    if (e != cudaSuccess) return cuda_fail(e, "readout launch");
    if ((e = cudaEventRecord(S->ro_done[bsel], S->lo)) != cudaSuccess) return cuda_fail(e, "event record");
    used[bsel] = true;
  }
  // the caller's stream resumes after the last scan and every read-out
  if ((e = cudaEventRecord(S->scan_done[0], S->hi)) != cudaSuccess) return cuda_fail(e, "event record");
  if ((e = cudaStreamWaitEvent(st, S->scan_done[0], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  for (int i = 0; i < 2; ++i)
    if (used[i] && (e = cudaStreamWaitEvent(st, S->ro_done[i], 0)) != cudaSuccess) return cuda_fail(e, "stream wait");
  return ok();
}

dla_status dla_forward(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv, const void* q,
                       const void* k, const void* v, const float* lam, void* o, const dla_cache* cache,
                       uint8_t* boundary, int32_t* merge_log, void* workspace, size_t ws_bytes, void* stream) {
  return forward_impl(p, in_dtype, B, T, H, dk, dv, q, k, v, lam, o, cache, boundary, merge_log, workspace, ws_bytes,
                      stream, nullptr);
}

dla_status dla_forward_varlen(const dla_params* p, dla_dtype in_dtype, int B, int max_seqlen, long long total_tokens,
                              const int32_t* cu_seqlens, int H, int dk, int dv, const void* q, const void* k,
                              const void* v, const float* lam, void* o, const dla_cache* cache, uint8_t* boundary,
                              int32_t* merge_log, void* workspace, size_t ws_bytes, void* stream) {
  const Varlen vl{cu_seqlens, total_tokens};
  return forward_impl(p, in_dtype, B, max_seqlen, H, dk, dv, q, k, v, lam, o, cache, boundary, merge_log, workspace,
                      ws_bytes, stream, nullptr, &vl);
}

// Device buffers of dla_forward_host at the end of its workspace: q, k, v,
// lambda, o (each 256-byte aligned); the forward pass's workspace before them.
struct HostBuffers {
  size_t q, k, v, lam, o, total;
};
static HostBuffers host_buffers(const dla_params* p, int B, int T, int H, int d, dla_dtype in_dtype, int with_output) {
  HostBuffers hb;
  const size_t n = (size_t)B * T * H * d, elt = (in_dtype == DLA_BF16) ? 2 : 4;
  const size_t oelt = (p->out_dtype == DLA_BF16) ? 2 : 4;
  size_t off = 0;
  hb.k = off;   off = align256(off + n * elt);
  hb.v = off;   off = align256(off + n * elt);
  hb.q = off;   if (with_output) off = align256(off + n * elt);
  hb.lam = off; if (with_output) off = align256(off + (size_t)B * T * H * p->capacity * sizeof(float));
  hb.o = off;   if (with_output) off = align256(off + n * oelt);
  hb.total = off;
  return hb;
}

size_t dla_forward_host_workspace(const dla_params* p, int B, int T, int H, int dk, int dv, dla_dtype in_dtype,
                                  int with_output) {
  if (check_params(p) != DLA_OK || check_shape(dk, dv) != DLA_OK || B < 1 || T < 1 || H < 1) return 0;
  return host_buffers(p, B, T, H, dk, in_dtype, with_output).total +
         dla_forward_workspace(p, B, T, H, dk, dv, in_dtype, with_output);
}

dla_status dla_forward_host(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv,
                            const void* q, const void* k, const void* v, const float* lam, void* o,
                            const dla_cache* cache, uint8_t* boundary, int32_t* merge_log, void* workspace,
                            size_t ws_bytes, void* stream) {
  dla_status s = check_params(p);
  if (s != DLA_OK) return s;
  if (in_dtype != DLA_BF16 && in_dtype != DLA_F32) return fail(DLA_ERR_INVALID_ARG, "bad in_dtype");
  if (B < 1 || T < 1 || H < 1) return fail(DLA_ERR_INVALID_ARG, "B, T, H must be >= 1");
  if ((s = check_shape(dk, dv)) != DLA_OK) return s;
  if (!k || !v) return fail(DLA_ERR_INVALID_ARG, "k and v must be non-NULL");
  if (o && !q) return fail(DLA_ERR_INVALID_ARG, "q must be non-NULL when o is requested");
  if (!workspace) return fail(DLA_ERR_WORKSPACE, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(DLA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const int d = dk;
  const bool with_output = (o != nullptr);
  const HostBuffers hb = host_buffers(p, B, T, H, d, in_dtype, with_output);
  if (ws_bytes < hb.total) return fail(DLA_ERR_WORKSPACE, "workspace has %zu bytes, needs more than %zu", ws_bytes, hb.total);
  const size_t fw_bytes = (ws_bytes - hb.total) & ~(size_t)255;  // the forward pass's part, before the buffers
  char* bufs = (char*)workspace + fw_bytes;
  HostIO io;
  io.qh = with_output ? q : nullptr;
  io.kh = k;
  io.vh = v;
  io.lamh = with_output ? lam : nullptr;
  io.qd = bufs + hb.q;
  io.kd = bufs + hb.k;
  io.vd = bufs + hb.v;
  io.lamd = (float*)(bufs + hb.lam);
  io.elt = (in_dtype == DLA_BF16) ? 2 : 4;
  io.oh = with_output ? o : nullptr;
  io.oelt = (p->out_dtype == DLA_BF16) ? 2 : 4;
  void* od = with_output ? bufs + hb.o : nullptr;
  s = forward_impl(p, in_dtype, B, T, H, dk, dv, with_output ? io.qd : nullptr, io.kd, io.vd,
                   (with_output && lam) ? io.lamd : nullptr, od, cache, boundary, merge_log, workspace, fw_bytes,
                   stream, &io);
  if (s != DLA_OK) return s;
  if (with_output && !io.o_streamed) {
    const size_t ob = (size_t)B * T * H * d * ((p->out_dtype == DLA_BF16) ? 2 : 4);
    const cudaError_t e = cudaMemcpyAsync(o, od, ob, cudaMemcpyDeviceToHost, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "output copy");
  }
  return ok();
}

dla_status dla_decode_step(const dla_params* p, const dla_cache* cache, dla_dtype in_dtype, const void* q,
                           const void* k, const void* v, const float* lam, void* o, uint8_t* boundary,
                           int32_t* merge_idx, void* stream) {
  dla_status s = check_params(p);
  if (s != DLA_OK) return s;
  if (in_dtype != DLA_BF16 && in_dtype != DLA_F32) return fail(DLA_ERR_INVALID_ARG, "bad in_dtype");
  if (!cache) return fail(DLA_ERR_INVALID_ARG, "cache is NULL");
  if ((s = check_shape(cache->dk, cache->dv)) != DLA_OK) return s;
  if ((s = check_cache(cache, cache->B, cache->H, p->capacity, cache->dk)) != DLA_OK) return s;
  if (p->capacity > dla::kMaxC)
    return fail(DLA_ERR_UNSUPPORTED, "dla_decode_step takes capacities up to %d", dla::kMaxC);
  if (!q || !k || !v || !o) return fail(DLA_ERR_INVALID_ARG, "q, k, v and o must be non-NULL");
  if (lam && !aligned(lam, 4)) return fail(DLA_ERR_INVALID_ARG, "lambda must be 4-byte aligned");
  dla::DecodeArgs da;
  memset(&da, 0, sizeof(da));
  da.q = q; da.k = k; da.v = v; da.lam = lam; da.o = o;
  da.out_bf16 = (p->out_dtype == DLA_BF16);
  da.B = cache->B; da.H = cache->H; da.C = cache->C;
  da.sp.tau = p->tau; da.sp.eps = p->eps; da.sp.rms_eps = p->rms_eps; da.sp.score_mode = p->score_mode;
  dla::finish_score_params(da.sp);
  da.states = cache->states; da.slot = cache->slot; da.n = cache->n; da.ibar = cache->ibar; da.m = cache->m;
  da.boundary = boundary; da.merge_idx = merge_idx;
  cudaError_t e = status_word((cudaStream_t)stream, &da.status);
  if (e != cudaSuccess) return cuda_fail(e, "status word");
  e = timed(DLA_K_DECODE, (cudaStream_t)stream,
                        [&] { return dla::launch_decode(da, cache->dk, in_dtype == DLA_BF16, (cudaStream_t)stream); });
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  return ok();
}

size_t dla_backward_workspace(const dla_params* p, int B, int T, int H, int dk, int dv, dla_dtype in_dtype) {
  if (!p || B < 1 || T < 1 || H < 1 || dk < 1 || dv < 1 || in_dtype != DLA_BF16) return 0;
  return 256 + align256(dla::backward_slot_bytes((int)((long long)B * H), T));
}

dla_status dla_backward(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv, const void* q,
                        const void* k, const void* v, const float* lam, const uint8_t* boundary,
                        const int32_t* merge_log, const float* grad_o, float* grad_q, float* grad_k, float* grad_v,
                        float* grad_lam, void* workspace, size_t ws_bytes, void* stream) {
  dla_status s = check_params(p);
  if (s != DLA_OK) return s;
  if (in_dtype != DLA_BF16 && in_dtype != DLA_F32) return fail(DLA_ERR_INVALID_ARG, "bad in_dtype");
  if (in_dtype != DLA_BF16) return fail(DLA_ERR_UNSUPPORTED, "dla_backward takes bf16 q, k, v");
  if (B < 1 || T < 1 || H < 1) return fail(DLA_ERR_INVALID_ARG, "B, T, H must be >= 1");
  if ((s = check_shape(dk, dv)) != DLA_OK) return s;
  if ((long long)B * H > 65535) return fail(DLA_ERR_UNSUPPORTED, "B * H must be at most 65535");
  if ((long long)B * T * H * dk >= (1LL << 40)) return fail(DLA_ERR_UNSUPPORTED, "tensor too large");
  if (p->from_cache) return fail(DLA_ERR_UNSUPPORTED, "dla_backward starts from an empty cache (from_cache = 0)");
  if (p->capacity > dla::kMaxC) return fail(DLA_ERR_UNSUPPORTED, "dla_backward takes capacities up to %d", dla::kMaxC);
  if (p->seq_lens) return fail(DLA_ERR_UNSUPPORTED, "dla_backward takes whole rows (seq_lens = NULL)");
  if (!q || !k || !v || !boundary || !merge_log || !grad_o || !grad_q || !grad_k || !grad_v)
    return fail(DLA_ERR_INVALID_ARG, "q, k, v, boundary, merge_log, grad_o, grad_q, grad_k, grad_v must be non-NULL");
  const void* a16[] = {q, k, v, grad_o, grad_q, grad_k, grad_v};
  for (const void* x : a16)
    if (!aligned(x, 16)) return fail(DLA_ERR_INVALID_ARG, "q, k, v and the gradients of o, q, k, v must be 16-byte aligned");
  if ((lam && !aligned(lam, 4)) || (grad_lam && !aligned(grad_lam, 4)))
    return fail(DLA_ERR_INVALID_ARG, "lambda and its gradient must be 4-byte aligned");
  if (!workspace) return fail(DLA_ERR_WORKSPACE, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(DLA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const size_t need = dla_backward_workspace(p, B, T, H, dk, dv, in_dtype);
  if (ws_bytes < need) return fail(DLA_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", ws_bytes, need);
  cudaStream_t st = (cudaStream_t)stream;
  char* ws = (char*)workspace;
  int32_t* word = nullptr;
  cudaError_t e = status_word(st, &word);
  if (e != cudaSuccess) return cuda_fail(e, "status word");
  dla::BackwardArgs ba;
  memset(&ba, 0, sizeof(ba));
  ba.q = q; ba.k = k; ba.v = v; ba.lam = lam; ba.g = grad_o;
  ba.boundary = boundary; ba.merge_log = merge_log;
  ba.dq = grad_q; ba.dk = grad_k; ba.dv = grad_v; ba.dlam = grad_lam;
  ba.B = B; ba.T = T; ba.H = H; ba.C = p->capacity;
  ba.status = (int32_t*)ws;
  ba.evt = (int32_t*)(ws + 256);
  ba.firsts = ba.evt + (size_t)B * H * T;
  if ((e = cudaMemsetAsync(ws, 0, 2 * sizeof(int32_t), st)) != cudaSuccess) return cuda_fail(e, "status reset");
  if ((e = timed(DLA_K_BACKWARD, st, [&] { return dla::launch_backward_slots(ba, st); })) != cudaSuccess)
    return cuda_fail(e, "backward slot lists launch");
  if ((e = timed(DLA_K_BACKWARD, st, [&] { return dla::launch_backward_dkv(ba, dk, st); })) != cudaSuccess)
    return cuda_fail(e, "backward dK, dV launch");
  if ((e = timed(DLA_K_BACKWARD, st, [&] { return dla::launch_backward_dq(ba, dk, st); })) != cudaSuccess)
    return cuda_fail(e, "backward dQ launch");
  e = timed(DLA_K_STATUS, st, [&] {
    status_fold_kernel<<<1, 1, 0, st>>>((const int32_t*)ws, word);
    return cudaGetLastError();
  });
  if (e != cudaSuccess) return cuda_fail(e, "status fold launch");
  return ok();
}

}  // extern "C"
