// bmlp_api.cu -- host side of the C-ABI declared in include/bmlp.h.
//
// One training mini-batch is one event-draw launch, L forward launches, one
// local-classifier + selection launch and one update launch.  All of them read
// the batch index s and the step counter t from a device-resident control block
// that the update kernel advances, so captured CUDA graphs (of eight steps, or
// one) replay step after step with no host work between steps.  Batch pointers
// live in a device-resident parameter block that a stream-ordered copy
// refreshes at the start of a call.  Each entry point that launches work opens
// an NVTX range named after it (header-only NVTX v3: a no-op unless a tracing
// tool is attached).
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstddef>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "bmlp_internal.cuh"
#include "update_common.cuh"

using namespace bk;

namespace {

thread_local std::string g_create_error;

// Process-wide accounting of the memory the library holds (every handle's
// device buffers and pinned host block), and the one-shot injected failure of
// the n-th allocation from the moment bmlp_debug_fail_alloc armed it.
std::atomic<int64_t> g_live_allocs{0}, g_live_bytes{0};
std::atomic<int64_t> g_fail_at{0}, g_alloc_seq{0};

// True when this allocation is the armed one (the injection then disarms).
bool injected_alloc_failure() {
  if (g_fail_at.load() <= 0) return false;
  const int64_t seq = ++g_alloc_seq;
  int64_t at = g_fail_at.load();
  return seq == at && g_fail_at.compare_exchange_strong(at, 0);
}

// NVTX range for the lifetime of an entry point call.
struct TraceRange {
  explicit TraceRange(const char* name) { nvtxRangePushA(name); }
  ~TraceRange() { nvtxRangePop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

enum ProfKind { kProfTrainFwd = 0, kProfCls = 1, kProfUpd = 2, kProfEvalFwd = 3, kProfOut = 4,
                kProfCopy = 5, kProfEvents = 6, kProfKinds = 7 };

}  // namespace

struct bmlp {
  int device = 0;
  int L = 0, c = 0, h_max = 0, bs = 0, r_num = 0, r_den = 1, fwd_impl = BMLP_FWD_POPC;
  int group_mode = BMLP_GROUPS_CONTIGUOUS, max_K = 0;  // group membership (Sec. 4.3), widest layer
  uint64_t seed = 0;
  std::vector<int> K, gamma;
  double p_r = 0.5;
  int64_t epoch_n = 0;  // patterns since the last epoch end
  int64_t t_host = 0;   // host mirror of ctrl->t
  StepParams hp{};      // host copy of the parameter block
  StepParams* dP = nullptr;
  Ctrl* dCtrl = nullptr;
  RTables* dRT = nullptr;
  std::vector<void*> allocs;
  int64_t held_bytes = 0;  // device bytes in allocs (+ the pinned host block)
  // evaluation scratch (grown on demand)
  uint64_t* evA[2] = {nullptr, nullptr};
  int64_t evCap = 0;
  // staging for host batches
  uint64_t* stX = nullptr;
  int32_t* stY = nullptr;
  int32_t* stOut = nullptr;
  int64_t stCap = 0;
  unsigned long long* hostPinned = nullptr;  // [4] D2H landing zone
  // graph of one training step
  cudaGraphExec_t stepExec = nullptr;   // one mini-batch step
  cudaGraphExec_t multiExec = nullptr;  // kGraphSteps consecutive steps
  cudaStream_t capStream = nullptr;
  cudaStream_t sideStream = nullptr;  // the event-draw branch of the step graph
  cudaEvent_t evFork = nullptr, evJoin = nullptr;
  int updCtas = 0;
  size_t updSmem = 0;
  // profiling
  bool profiling = false;       // events around the kernels being enqueued now
  int32_t profEvery = 0;        // 0 off, 1 every mini-batch, S every S-th mini-batch
  std::vector<cudaEvent_t> evPool;
  size_t evUsed = 0;
  std::vector<std::pair<int, size_t>> evPairs;  // (kind, index of start event)
  int64_t profN[kProfKinds] = {0};
  double profMs[kProfKinds] = {0};
  int64_t launches = 0;
  std::string err;
};

namespace {

int fail(bmlp_t* h, int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  if (h) h->err = buf; else g_create_error = buf;
  return code;
}

int cuda_fail(bmlp_t* h, cudaError_t e, const char* what) {
  return fail(h, e == cudaErrorMemoryAllocation ? BMLP_ENOMEM : BMLP_ECUDA, "%s: %s", what,
              cudaGetErrorString(e));
}

#define CK(h, call)                                   \
  do {                                                \
    cudaError_t e_ = (call);                          \
    if (e_ != cudaSuccess) return cuda_fail(h, e_, #call); \
  } while (0)

template <typename T>
int dalloc(bmlp_t* h, T** p, size_t count) {
  void* q = nullptr;
  const size_t bytes = count * sizeof(T) > 0 ? count * sizeof(T) : 16;
  if (injected_alloc_failure()) return fail(h, BMLP_ENOMEM, "cudaMalloc of %zu bytes failed (injected)", bytes);
  cudaError_t e = cudaMalloc(&q, bytes);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaMalloc");
  h->allocs.push_back(q);
  h->held_bytes += (int64_t)bytes;
  g_live_allocs += 1;
  g_live_bytes += (int64_t)bytes;
  *p = static_cast<T*>(q);
  return BMLP_OK;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int words_of(int K) { return (K + 63) / 64; }

// thr(x) of the reinforcement sampler: the integer T with (V < T) <=> (V / 2^32 < x)
// for every 32-bit V.
uint64_t sampler_thr(double x) {
  if (!(x > 0.0)) return 0;
  if (x >= 1.0) return (uint64_t)1 << 32;
  return (uint64_t)std::ceil(x * 4294967296.0);
}

// Sampler thresholds of a block of n (1..64) inputs at probability q.
void block_tables(double q, int n, unsigned long long* any, unsigned long long* first,
                  unsigned long long* gap) {
  if (q > 1.0) q = 1.0;
  const double s = 1.0 - q;
  double pw[65];
  pw[0] = 1.0;
  for (int m = 1; m <= n; ++m) pw[m] = pw[m - 1] * s;
  const double p_any = 1.0 - pw[n];
  *any = sampler_thr(p_any);
  for (int j = 0; j < n; ++j) first[j] = sampler_thr((1.0 - pw[j + 1]) / p_any);
  if (gap)
    for (int g = 0; g + 1 < n; ++g) gap[g] = sampler_thr(1.0 - pw[g + 1]);
}

double reinforce_q(double p_r, int K) { return p_r * std::sqrt(2.0 / (M_PI * (double)K)); }

int upload_thresholds(bmlp_t* h, cudaStream_t st) {
  std::vector<RTables> rt((size_t)h->L);
  for (int l = 1; l <= h->L; ++l) {
    RTables& R = rt[(size_t)l - 1];
    std::memset(&R, 0, sizeof(R));
    const double q = reinforce_q(h->p_r, h->K[l]);
    block_tables(q, 64, &R.any[0], R.first[0], R.gap);
    const int tail = h->K[l - 1] % 64;
    if (tail) block_tables(q, tail, &R.any[1], R.first[1], nullptr);
  }
  CK(h, cudaMemcpyAsync(h->dRT, rt.data(), sizeof(RTables) * (size_t)h->L, cudaMemcpyHostToDevice,
                        st));
  CK(h, cudaStreamSynchronize(st));  // rt is a host temporary
  return BMLP_OK;
}

// event-bracketed launch in profiling mode
cudaEvent_t next_event(bmlp_t* h) {
  if (h->evUsed == h->evPool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->evPool.push_back(e);
  }
  return h->evPool[h->evUsed++];
}

void prof_begin(bmlp_t* h, int kind, cudaStream_t st) {
  if (!h->profiling) return;
  cudaEvent_t a = next_event(h);
  cudaEvent_t b = next_event(h);
  if (!a || !b) return;
  h->evPairs.push_back({kind, h->evUsed - 2});
  cudaEventRecord(a, st);
}

void prof_end(bmlp_t* h, cudaStream_t st) {
  if (!h->profiling || h->evPairs.empty()) return;
  cudaEventRecord(h->evPool[h->evPairs.back().second + 1], st);
}

int prof_collect(bmlp_t* h, cudaStream_t st) {
  if (!h->profiling || h->evPairs.empty()) return BMLP_OK;
  CK(h, cudaStreamSynchronize(st));
  for (auto& pr : h->evPairs) {
    float ms = 0.f;
    CK(h, cudaEventElapsedTime(&ms, h->evPool[pr.second], h->evPool[pr.second + 1]));
    h->profMs[pr.first] += ms;
    h->profN[pr.first] += 1;
  }
  h->evPairs.clear();
  h->evUsed = 0;
  return BMLP_OK;
}

// Enqueue the kernels of one training mini-batch on `st`.  The reinforcement
// events depend only on (seed, layer, neuron, step, p_r): when `fork` is set
// (graph capture) their kernel runs on a side stream next to the forward
// passes, which leave most of every SM idle, and joins before the update;
// otherwise it runs first on `st`.
// Mini-batch steps per captured training graph (a shorter run, or one that
// has sampled steps in the way, uses the one-step graph).
constexpr int kGraphSteps = 8;

// One mini-batch step.  fork: the graph form (event draws on a branch,
// programmatic dependent launches); chained: the step follows another step in
// the same graph, so its first forward is a dependent of that step's update.
int enqueue_step(bmlp_t* h, cudaStream_t st, bool fork, bool chained = false) {
  if (!fork) {
    prof_begin(h, kProfEvents, st);
    launch_r_events((unsigned)h->hp.ev_ctas_total, st, h->dP, h->hp.key0, h->hp.key1);
    prof_end(h, st);
  }
  // one hidden layer whose forward pass leaves most SMs free (at most 64
  // CTAs): the event draws start with the step
  const bool early = h->L == 1 && ((h->K[1] + 255) / 256) * 4 <= 64;
  for (int l = 1; l <= h->L; ++l) {
    if (fork && l == (early ? 1 : 2)) {
      // otherwise fork after the first forward pass: its CTAs hold the SMs,
      // and the event draws and the second pass become ready together
      CK(h, cudaEventRecord(h->evFork, st));
      CK(h, cudaStreamWaitEvent(h->sideStream, h->evFork, 0));
      launch_r_events((unsigned)h->hp.ev_ctas_total, h->sideStream, h->dP, h->hp.key0, h->hp.key1);
      CK(h, cudaEventRecord(h->evJoin, h->sideStream));
    }
    prof_begin(h, kProfTrainFwd, st);
    if (h->fwd_impl == BMLP_FWD_TCGEN05)
      CK(h, launch_train_forward_tc(h->K[l], st, fork && (l > 1 || chained), h->dP, l));
    else
      k_train_forward<<<train_forward_grid(h->bs, h->K[l]), train_forward_block(), 0, st>>>(h->dP, l);
    prof_end(h, st);
  }
  if (h->group_mode == BMLP_GROUPS_RESHUFFLED) {
    // this step's partition (keyed by the step counter) before the selection
    CK(h, launch_group_order(h->L, h->max_K, true, st, h->dP));
  }
  prof_begin(h, kProfCls, st);
  // inside the step graph each kernel after the first is launched as a
  // programmatic dependent of the one before it (launch and prologue overlap
  // the previous kernel's tail); the event-draw branch joins with a full edge
  CK(h, launch_kernel(k_cls_select, dim3((unsigned)h->bs, (unsigned)h->L), dim3(kClsThreads), 0, st,
                      fork && h->fwd_impl == BMLP_FWD_TCGEN05, h->dP));
  prof_end(h, st);
  if (fork && h->L == 1 && !early) {
    CK(h, cudaEventRecord(h->evFork, st));
    CK(h, cudaStreamWaitEvent(h->sideStream, h->evFork, 0));
    launch_r_events((unsigned)h->hp.ev_ctas_total, h->sideStream, h->dP, h->hp.key0, h->hp.key1);
    CK(h, cudaEventRecord(h->evJoin, h->sideStream));
  }
  if (fork) CK(h, cudaStreamWaitEvent(st, h->evJoin, 0));
  prof_begin(h, kProfUpd, st);
  CK(h, launch_update_ws(h->hp.nplanes, h->h_max, h->bs, (unsigned)h->updCtas, st, fork, h->dP));
  prof_end(h, st);
  CK(h, cudaGetLastError());
  return BMLP_OK;
}

// Capture `steps` consecutive mini-batch steps into one executable graph.
int capture_steps(bmlp_t* h, int steps, cudaGraphExec_t* exec) {
  cudaGraph_t g = nullptr;
  CK(h, cudaStreamBeginCapture(h->capStream, cudaStreamCaptureModeThreadLocal));
  const bool prof = h->profiling;
  h->profiling = false;
  int rc = BMLP_OK;
  for (int i = 0; i < steps && rc == BMLP_OK; ++i) rc = enqueue_step(h, h->capStream, true, i > 0);
  h->profiling = prof;
  cudaError_t e = cudaStreamEndCapture(h->capStream, &g);
  if (rc != BMLP_OK) {
    if (g) cudaGraphDestroy(g);
    return rc;
  }
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaStreamEndCapture");
  e = cudaGraphInstantiate(exec, g, cudaGraphInstantiateFlagUseNodePriority);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return cuda_fail(h, e, "cudaGraphInstantiate");
  return BMLP_OK;
}

int ensure_graph(bmlp_t* h) {
  if (h->stepExec && h->multiExec) return BMLP_OK;
  // the forward chain is captured at the highest stream priority and the
  // event-draw branch at the lowest, so that the block scheduler places
  // forward CTAs first and the event draws fill the remaining room
  int prio_low = 0, prio_high = 0;
  CK(h, cudaDeviceGetStreamPriorityRange(&prio_low, &prio_high));
  if (!h->capStream)
    CK(h, cudaStreamCreateWithPriority(&h->capStream, cudaStreamNonBlocking, prio_high));
  if (!h->sideStream)
    CK(h, cudaStreamCreateWithPriority(&h->sideStream, cudaStreamNonBlocking, prio_low));
  if (!h->evFork) CK(h, cudaEventCreateWithFlags(&h->evFork, cudaEventDisableTiming));
  if (!h->evJoin) CK(h, cudaEventCreateWithFlags(&h->evJoin, cudaEventDisableTiming));
  int rc;
  if (!h->stepExec && (rc = capture_steps(h, 1, &h->stepExec)) != BMLP_OK) return rc;
  if (!h->multiExec && (rc = capture_steps(h, kGraphSteps, &h->multiExec)) != BMLP_OK) return rc;
  return BMLP_OK;
}

// Train on n device-resident patterns.
int run_steps(bmlp_t* h, const uint64_t* xd, const int32_t* yd, int64_t n, cudaStream_t st) {
  h->hp.x = xd;
  h->hp.y = yd;
  h->hp.n = n;
  const size_t head = offsetof(StepParams, x);
  CK(h, cudaMemcpyAsync(reinterpret_cast<char*>(h->dP) + head, reinterpret_cast<char*>(&h->hp) + head,
                        sizeof(StepParams) - head, cudaMemcpyHostToDevice, st));
  CK(h, cudaMemsetAsync(&h->dCtrl->s, 0, sizeof(uint32_t), st));
  const int64_t steps = (n + h->bs - 1) / h->bs;
  if (h->profEvery != 1) {
    int rc = ensure_graph(h);
    if (rc != BMLP_OK) return rc;
  }
  auto sampled = [&](int64_t s) {
    return h->profEvery > 0 && ((h->t_host + s) % h->profEvery) == 0;
  };
  for (int64_t s = 0; s < steps;) {
    // sampled mini-batches are launched kernel by kernel between CUDA events;
    // the others as graphs of kGraphSteps steps, or of one step
    h->profiling = sampled(s);
    if (h->profiling) {
      int rc = enqueue_step(h, st, false);
      if (rc != BMLP_OK) return rc;
      ++s;
      continue;
    }
    bool multi = s + kGraphSteps <= steps;
    for (int64_t i = 1; multi && i < kGraphSteps; ++i) multi = !sampled(s + i);
    CK(h, cudaGraphLaunch(multi ? h->multiExec : h->stepExec, st));
    s += multi ? kGraphSteps : 1;
  }
  h->profiling = h->profEvery > 0;
  h->launches += steps * (h->L + 3 + (h->group_mode == BMLP_GROUPS_RESHUFFLED ? 1 : 0));
  h->t_host += steps;
  return BMLP_OK;
}

int ensure_staging(bmlp_t* h, int64_t rows) {
  if (rows <= h->stCap) return BMLP_OK;
  int rc;
  if ((rc = dalloc(h, &h->stX, (size_t)rows * h->hp.nw0)) != BMLP_OK) return rc;
  if ((rc = dalloc(h, &h->stY, (size_t)rows)) != BMLP_OK) return rc;
  if ((rc = dalloc(h, &h->stOut, (size_t)rows)) != BMLP_OK) return rc;
  h->stCap = rows;
  return BMLP_OK;
}

int ensure_eval(bmlp_t* h, int64_t rows) {
  if (rows <= h->evCap) return BMLP_OK;
  int nwmax = 0;
  for (int l = 1; l <= h->L; ++l) nwmax = std::max(nwmax, words_of(h->K[l]));
  int rc;
  if ((rc = dalloc(h, &h->evA[0], (size_t)rows * nwmax)) != BMLP_OK) return rc;
  if ((rc = dalloc(h, &h->evA[1], (size_t)rows * nwmax)) != BMLP_OK) return rc;
  h->evCap = rows;
  return BMLP_OK;
}

constexpr int64_t kEvalChunk = 65536;
constexpr int64_t kStageRows = 65536;

}  // namespace

// ---------------------------------------------------------------------------
extern "C" {

int32_t bmlp_gamma_rule(int32_t K) {
  if (K < 1) return -1;
  int32_t best = -1, bestd = 0;
  for (int32_t g = 1; g <= K; ++g) {
    if (K % g) continue;
    const int32_t d = g < 75 ? 75 - g : (g > 105 ? g - 105 : 0);
    if (best < 0 || d < bestd || (d == bestd && g > best)) {
      best = g;
      bestd = d;
    }
  }
  return best;
}

int bmlp_reinforce_tables(double p_r, int32_t K, int32_t n, uint64_t* any_out,
                          uint64_t* first_out, uint64_t* gap_out) {
  if (K < 1 || n < 1 || n > 64 || !any_out || !first_out || !gap_out) return BMLP_EINVAL;
  unsigned long long a = 0, f[64], g[64];
  block_tables(reinforce_q(p_r, K), n, &a, f, g);
  *any_out = a;
  for (int j = 0; j < n; ++j) first_out[j] = f[j];
  for (int j = 0; j + 1 < n; ++j) gap_out[j] = g[j];
  return BMLP_OK;
}

const char* bmlp_last_error(const bmlp_t* h) {
  return h ? h->err.c_str() : g_create_error.c_str();
}

int bmlp_create(const int32_t* widths, int32_t n_widths, int32_t classes, int16_t h_max,
                uint64_t seed, const bmlp_hparams* hpin, bmlp_t** out) {
  TraceRange trace("bmlp_create");
  g_create_error.clear();
  if (!out) return fail(nullptr, BMLP_EINVAL, "out is NULL");
  *out = nullptr;
  if (!widths) return fail(nullptr, BMLP_EINVAL, "widths is NULL");
  if (n_widths < 2 || n_widths > BMLP_MAX_LAYERS + 1)
    return fail(nullptr, BMLP_EINVAL, "n_widths must be in 2..%d", BMLP_MAX_LAYERS + 1);
  for (int i = 0; i < n_widths; ++i)
    if (widths[i] < 1 || widths[i] > 32767)  // |z| <= K_{l-1} must fit the int16 Z buffer
      return fail(nullptr, BMLP_EINVAL, "width %d out of range (1..32767)", i);
  if (classes < 2 || classes > BMLP_MAX_CLASSES)
    return fail(nullptr, BMLP_EINVAL, "classes must be in 2..%d", BMLP_MAX_CLASSES);
  if (h_max < 1 || h_max > 16383 || (h_max % 2) == 0)
    return fail(nullptr, BMLP_EINVAL, "h_max must be odd and in 1..16383");
  bmlp_hparams hp{};
  if (hpin) hp = *hpin;
  const int bs = hp.bs == 0 ? 100 : hp.bs;
  if (bs < 1 || bs > BMLP_MAX_BS) return fail(nullptr, BMLP_EINVAL, "bs must be in 1..%d", BMLP_MAX_BS);
  int r_num = hp.r_num, r_den = hp.r_den;
  if (r_den == 0) { r_num = 1; r_den = 4; }
  if (r_den < 0 || r_num < 0) return fail(nullptr, BMLP_EINVAL, "r must be non-negative");
  const double p_r0 = hp.p_r0 < 0 ? 0.5 : hp.p_r0;
  if (!(p_r0 >= 0.0) || !std::isfinite(p_r0)) return fail(nullptr, BMLP_EINVAL, "p_r0 invalid");
  int fwd = hp.fwd_impl;
  if (fwd == BMLP_FWD_AUTO) fwd = bs <= 128 ? BMLP_FWD_TCGEN05 : BMLP_FWD_POPC;
  if (fwd != BMLP_FWD_POPC && fwd != BMLP_FWD_TCGEN05)
    return fail(nullptr, BMLP_EINVAL, "fwd_impl %d not available", hp.fwd_impl);
  if (fwd == BMLP_FWD_TCGEN05 && bs > 128)
    return fail(nullptr, BMLP_EINVAL, "fwd_impl TCGEN05 needs bs <= 128");
  const int L = n_widths - 1;
  const int group_mode = hp.group_mode;
  if (group_mode < BMLP_GROUPS_CONTIGUOUS || group_mode > BMLP_GROUPS_RESHUFFLED)
    return fail(nullptr, BMLP_EINVAL, "group_mode must be 0, 1 or 2");
  int max_K = 0;
  for (int l = 1; l <= L; ++l) max_K = std::max(max_K, (int)widths[l]);
  if (group_mode != BMLP_GROUPS_CONTIGUOUS && max_K > 16384)
    return fail(nullptr, BMLP_EINVAL, "random group membership needs every K_l <= 16384");
  std::vector<int> gam(L + 1, 0);
  for (int l = 1; l <= L; ++l) {
    const int g = hp.gamma ? hp.gamma[l - 1] : bmlp_gamma_rule(widths[l]);
    if (g < 1 || widths[l] % g) return fail(nullptr, BMLP_EINVAL, "gamma of layer %d must divide K_l", l);
    gam[l] = g;
  }
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
    (void)cudaGetLastError();
    return fail(nullptr, BMLP_ENODEV, "no CUDA device");
  }

  bmlp_t* h = new (std::nothrow) bmlp_t();
  if (!h) return fail(nullptr, BMLP_ENOMEM, "host allocation failed");
  cudaGetDevice(&h->device);
  cudaDeviceProp prop;
  cudaFuncAttributes fa;
  if (cudaGetDeviceProperties(&prop, h->device) != cudaSuccess || prop.major != 10 ||
      update_kernel_image(&fa) != cudaSuccess) {
    (void)cudaGetLastError();
    delete h;
    return fail(nullptr, BMLP_ENODEV, "device has no sm_103a kernel image (needs a GB300)");
  }
  h->L = L; h->c = classes; h->h_max = h_max; h->bs = bs; h->r_num = r_num; h->r_den = r_den;
  h->fwd_impl = fwd; h->seed = seed; h->p_r = p_r0;
  h->group_mode = group_mode; h->max_K = max_K;
  h->K.assign(widths, widths + n_widths);
  h->gamma = gam;

  auto bail = [&](int rc) { std::string m = h->err; bmlp_destroy(h); g_create_error = m; return rc; };
  int rc;
  StepParams& P = h->hp;
  std::memset(&P, 0, sizeof(P));
  P.L = L; P.c = classes; P.bs = bs; P.h_max = h_max; P.r_num = r_num; P.r_den = r_den;
  P.nw0 = words_of(widths[0]);
  P.nbits = upd::bits_of(h_max);
  P.nplanes = upd::planes_of(P.nbits);
  P.key0 = (uint32_t)(seed & 0xffffffffu);
  P.key1 = (uint32_t)(seed >> 32);
  int ev_cta = 0, rows_total = 0;
  for (int l = 1; l <= L; ++l) {
    DevLayer& D = P.layer[l - 1];
    D.Kin = h->K[l - 1]; D.Kout = h->K[l];
    D.nw_in = words_of(D.Kin); D.nw_out = words_of(D.Kout);
    D.ngrp = (D.Kin + 31) / 32;
    D.ldh = (D.ngrp * P.nplanes + 3) & ~3;
    D.gamma = gam[l]; D.G = D.Kout / D.gamma;
    D.row_base = rows_total;
    rows_total += D.Kout;
    D.ev_cta_base = ev_cta;
    ev_cta += (D.Kout + kEvRowsPerCta - 1) / kEvRowsPerCta;
    D.nblk = (D.Kin + 63) / 64;
    D.ev_stride = (D.nblk + 1) & ~1;
    if ((rc = dalloc(h, &D.H, (size_t)D.Kout * D.ldh)) ||
        (rc = dalloc(h, &D.W, (size_t)D.Kout * D.nw_in)) ||
        (rc = dalloc(h, &D.PT, (size_t)classes * D.nw_out)) ||
        (rc = dalloc(h, &D.rho, (size_t)D.Kout * classes)) ||
        (rc = dalloc(h, &D.rhoT, (size_t)D.Kout * classes)) ||
        (rc = dalloc(h, &D.Z, (size_t)bs * D.Kout)) ||
        (rc = dalloc(h, &D.A, (size_t)bs * D.nw_out)) ||
        (rc = dalloc(h, &D.mark, (size_t)bs)) ||
        (rc = dalloc(h, &D.sel, (size_t)bs * D.G)) ||
        (rc = dalloc(h, &D.EV, (size_t)D.Kout * D.ev_stride)))
      return bail(rc);
    D.member = D.group_of = nullptr;
    if (group_mode != BMLP_GROUPS_CONTIGUOUS &&
        ((rc = dalloc(h, &D.member, (size_t)D.Kout)) || (rc = dalloc(h, &D.group_of, (size_t)D.Kout))))
      return bail(rc);
  }
  P.rows_total = rows_total;
  P.ev_ctas_total = ev_cta;
  P.nblk_max = 0;
  for (int l = 1; l <= L; ++l) P.nblk_max = std::max(P.nblk_max, (widths[l - 1] + 63) / 64);
  {
    // the update grid is persistent, one CTA per SM (its slot ring fills most
    // of the shared memory)
    h->updSmem = update_ws_smem(P.nplanes, bs);
    const cudaError_t ea = prepare_update_ws();
    if (ea != cudaSuccess) return bail(cuda_fail(h, ea, "update kernel shared memory attribute"));
    h->updCtas = prop.multiProcessorCount;
    P.upd_ctas_total = h->updCtas;
  }
  if ((rc = dalloc(h, &h->dP, 1)) || (rc = dalloc(h, &h->dCtrl, 1)) ||
      (rc = dalloc(h, &h->dRT, BMLP_MAX_LAYERS)))
    return bail(rc);
  P.ctrl = h->dCtrl;
  P.rt = h->dRT;
  if (injected_alloc_failure())
    return bail(fail(h, BMLP_ENOMEM, "cudaMallocHost failed (injected)"));
  if (cudaMallocHost(&h->hostPinned, 4 * sizeof(unsigned long long)) != cudaSuccess) {
    h->hostPinned = nullptr;
    return bail(fail(h, BMLP_ENOMEM, "cudaMallocHost failed"));
  }
  g_live_allocs += 1;
  g_live_bytes += (int64_t)(4 * sizeof(unsigned long long));
  // initial state (Alg. 1 l.2)
  for (int l = 1; l <= L; ++l) {
    DevLayer& D = P.layer[l - 1];
    const int64_t n1 = (int64_t)D.Kout * D.ngrp;
    cudaMemsetAsync(D.H, 0, sizeof(uint32_t) * D.Kout * D.ldh);
    cudaMemsetAsync(D.W, 0, sizeof(uint64_t) * D.Kout * D.nw_in);
    k_init_hw<<<(unsigned)((n1 + 255) / 256), 256>>>(D.H, D.W, D.Kin, D.Kout, D.ldh, D.ngrp, P.nplanes,
                                                       l, P.key0, P.key1, h_max);
    const int64_t n2 = (int64_t)D.Kout * classes;
    k_init_rho<<<(unsigned)((n2 + 255) / 256), 256>>>(D.rho, D.Kout, classes, l, P.key0, P.key1);
    const int64_t n3 = (int64_t)classes * D.nw_out;
    k_pack_pt<<<(unsigned)((n3 + 255) / 256), 256>>>(D.rho, D.PT, D.Kout, classes, D.nw_out);
    k_transpose_rho<<<(unsigned)((n2 + 255) / 256), 256>>>(D.rho, D.rhoT, D.Kout, classes);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return bail(cuda_fail(h, e, "init kernels"));
  if (fwd == BMLP_FWD_TCGEN05 &&
      ((e = prepare_train_forward_tc()) != cudaSuccess || (e = prepare_forward_eval_tc()) != cudaSuccess))
    return bail(cuda_fail(h, e, "tcgen05 forward smem attribute"));
  if ((e = cudaMemset(h->dCtrl, 0, sizeof(Ctrl))) != cudaSuccess) return bail(cuda_fail(h, e, "memset"));
  if ((e = cudaMemcpy(h->dP, &P, sizeof(P), cudaMemcpyHostToDevice)) != cudaSuccess)
    return bail(cuda_fail(h, e, "param upload"));
  if ((rc = upload_thresholds(h, 0)) != BMLP_OK) return bail(rc);
  // the partition of step 0 (the fixed one, or the first redrawn one)
  if (group_mode != BMLP_GROUPS_CONTIGUOUS &&
      ((e = prepare_group_order(max_K)) != cudaSuccess ||
       (e = launch_group_order(L, max_K, false, 0, h->dP)) != cudaSuccess))
    return bail(cuda_fail(h, e, "group order"));
  if ((e = cudaDeviceSynchronize()) != cudaSuccess) return bail(cuda_fail(h, e, "init"));
  h->launches += 4 * L;
  *out = h;
  return BMLP_OK;
}

void bmlp_destroy(bmlp_t* h) {
  if (!h) return;
  cudaDeviceSynchronize();
  if (h->stepExec) cudaGraphExecDestroy(h->stepExec);
  if (h->multiExec) cudaGraphExecDestroy(h->multiExec);
  if (h->capStream) cudaStreamDestroy(h->capStream);
  if (h->sideStream) cudaStreamDestroy(h->sideStream);
  if (h->evFork) cudaEventDestroy(h->evFork);
  if (h->evJoin) cudaEventDestroy(h->evJoin);
  for (auto e : h->evPool) cudaEventDestroy(e);
  for (void* p : h->allocs) cudaFree(p);
  g_live_allocs -= (int64_t)h->allocs.size();
  g_live_bytes -= h->held_bytes;
  if (h->hostPinned) {
    cudaFreeHost(h->hostPinned);
    g_live_allocs -= 1;
    g_live_bytes -= (int64_t)(4 * sizeof(unsigned long long));
  }
  delete h;
}

int bmlp_train(bmlp_t* h, const uint64_t* x, const int32_t* labels, int64_t n, uint32_t flags,
               void* cuda_stream, int64_t* n_errors_out) {
  TraceRange trace("bmlp_train");
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (n < 0) return fail(h, BMLP_EINVAL, "n < 0");
  if (n > 0 && (!x || !labels)) return fail(h, BMLP_EINVAL, "x or labels is NULL");
  if ((n + h->bs - 1) / h->bs > 0xffffffffLL) return fail(h, BMLP_EINVAL, "n too large");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const bool want_count = n_errors_out != nullptr;
  if (want_count) {
    CK(h, cudaMemcpyAsync(&h->hostPinned[0], &h->dCtrl->err, sizeof(unsigned long long),
                          cudaMemcpyDeviceToHost, st));
  }
  int rc = BMLP_OK;
  if (n > 0) {
    const bool xdev = is_device_ptr(x), ydev = is_device_ptr(labels);
    if (xdev && ydev) {
      rc = run_steps(h, x, labels, n, st);
    } else {
      if (!ydev)
        for (int64_t i = 0; i < n; ++i)
          if (labels[i] < 0 || labels[i] >= h->c) return fail(h, BMLP_EINVAL, "label %lld out of range", (long long)i);
      const int64_t chunk = (kStageRows / h->bs) * h->bs;
      if ((rc = ensure_staging(h, chunk)) != BMLP_OK) return rc;
      for (int64_t s0 = 0; s0 < n && rc == BMLP_OK; s0 += chunk) {
        const int64_t m = std::min(chunk, n - s0);
        const uint64_t* xs = x + s0 * h->hp.nw0;
        const int32_t* ys = labels + s0;
        prof_begin(h, kProfCopy, st);
        if (!xdev) CK(h, cudaMemcpyAsync(h->stX, xs, sizeof(uint64_t) * m * h->hp.nw0, cudaMemcpyHostToDevice, st));
        if (!ydev) CK(h, cudaMemcpyAsync(h->stY, ys, sizeof(int32_t) * m, cudaMemcpyHostToDevice, st));
        prof_end(h, st);
        rc = run_steps(h, xdev ? xs : h->stX, ydev ? ys : h->stY, m, st);
      }
    }
    if (rc != BMLP_OK) return rc;
  }
  h->epoch_n += n;
  const bool epoch_end = (flags & BMLP_EPOCH_END) != 0;
  if (want_count || epoch_end) {
    CK(h, cudaMemcpyAsync(&h->hostPinned[1], &h->dCtrl->err, sizeof(unsigned long long),
                          cudaMemcpyDeviceToHost, st));
    CK(h, cudaMemcpyAsync(&h->hostPinned[2], &h->dCtrl->bad_labels, sizeof(unsigned long long),
                          cudaMemcpyDeviceToHost, st));
    CK(h, cudaMemcpyAsync(&h->hostPinned[3], &h->dCtrl->timeouts, sizeof(uint32_t),
                          cudaMemcpyDeviceToHost, st));
    CK(h, cudaStreamSynchronize(st));
    if ((uint32_t)h->hostPinned[3] != 0) {
      CK(h, cudaMemsetAsync(&h->dCtrl->timeouts, 0, sizeof(uint32_t), st));
      h->hostPinned[3] = 0;
      return fail(h, BMLP_ETIMEOUT, "a bounded device-side wait expired");
    }
    if (h->hostPinned[2] != 0) {
      CK(h, cudaMemsetAsync(&h->dCtrl->bad_labels, 0, sizeof(unsigned long long), st));
      return fail(h, BMLP_EINVAL, "%llu labels outside 0..c-1", (unsigned long long)h->hostPinned[2]);
    }
    if (want_count) *n_errors_out = (int64_t)(h->hostPinned[1] - h->hostPinned[0]);
    if (epoch_end) {
      const double E = h->epoch_n > 0 ? (double)h->hostPinned[1] / (double)h->epoch_n : 0.0;
      h->p_r = h->p_r * std::sqrt(E);
      h->epoch_n = 0;
      CK(h, cudaMemsetAsync(&h->dCtrl->err, 0, sizeof(unsigned long long), st));
      if ((rc = upload_thresholds(h, st)) != BMLP_OK) return rc;
    }
  }
  return prof_collect(h, st);
}

namespace {

// Forward-only evaluation of n patterns (Sec. 3.1).  every_layer: the argmax of
// a_l P_l of every layer l into out[(l-1) n + mu] (early exit); else of the
// last layer only into out[mu].
int predict_impl(bmlp_t* h, const uint64_t* x, int64_t n, int32_t* out, void* cuda_stream,
                 bool every_layer) {
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (n < 0) return fail(h, BMLP_EINVAL, "n < 0");
  if (n == 0) return BMLP_OK;
  if (!x || !out) return fail(h, BMLP_EINVAL, "x or labels_out is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const bool xdev = is_device_ptr(x), odev = is_device_ptr(out);
  int rc;
  const int64_t chunk = std::min<int64_t>(kEvalChunk, n);
  if ((rc = ensure_eval(h, chunk)) != BMLP_OK) return rc;
  if ((!xdev || !odev) && (rc = ensure_staging(h, kStageRows)) != BMLP_OK) return rc;
  const int nw0 = h->hp.nw0;
  for (int64_t s0 = 0; s0 < n; s0 += chunk) {
    const int64_t m = std::min(chunk, n - s0);
    const uint64_t* in = x + s0 * nw0;
    if (!xdev) {
      prof_begin(h, kProfCopy, st);
      CK(h, cudaMemcpyAsync(h->stX, in, sizeof(uint64_t) * m * nw0, cudaMemcpyHostToDevice, st));
      prof_end(h, st);
      in = h->stX;
    }
    int cur = 0;
    for (int l = 1; l <= h->L; ++l) {
      const DevLayer& D = h->hp.layer[l - 1];
      prof_begin(h, kProfEvalFwd, st);
      if (h->fwd_impl == BMLP_FWD_TCGEN05)
        launch_forward_eval_tc(in, m, D.nw_in, D.W, D.Kout, D.Kin, h->evA[cur], D.nw_out,
                               &h->dCtrl->timeouts, st);
      else
        k_forward_eval<<<eval_forward_grid(m, D.Kout), eval_forward_block(), 0, st>>>(
            in, m, D.nw_in, D.W, D.Kout, D.Kin, h->evA[cur], D.nw_out);
      prof_end(h, st);
      in = h->evA[cur];
      cur ^= 1;
      if (!every_layer && l < h->L) continue;
      // argmax of a_l P_l (lowest class on ties)
      int32_t* dst = out + (every_layer ? (int64_t)(l - 1) * n : 0) + s0;
      int32_t* o = odev ? dst : h->stOut;
      prof_begin(h, kProfOut, st);
      k_predict_out<<<(unsigned)((m + 7) / 8), 256, 0, st>>>(in, m, D.nw_out, D.PT, h->c, D.Kout, o);
      prof_end(h, st);
      CK(h, cudaGetLastError());
      h->launches += 1;
      if (!odev) {
        prof_begin(h, kProfCopy, st);
        CK(h, cudaMemcpyAsync(dst, h->stOut, sizeof(int32_t) * m, cudaMemcpyDeviceToHost, st));
        prof_end(h, st);
      }
    }
    h->launches += h->L;
  }
  if (!odev) {
    if (h->fwd_impl == BMLP_FWD_TCGEN05)
      CK(h, cudaMemcpyAsync(&h->hostPinned[3], &h->dCtrl->timeouts, sizeof(uint32_t),
                            cudaMemcpyDeviceToHost, st));
    CK(h, cudaStreamSynchronize(st));
    if (h->fwd_impl == BMLP_FWD_TCGEN05 && (uint32_t)h->hostPinned[3] != 0) {
      CK(h, cudaMemsetAsync(&h->dCtrl->timeouts, 0, sizeof(uint32_t), st));
      h->hostPinned[3] = 0;
      return fail(h, BMLP_ETIMEOUT, "a bounded device-side wait expired");
    }
  }
  return prof_collect(h, st);
}

}  // namespace

int bmlp_predict(bmlp_t* h, const uint64_t* x, int64_t n, int32_t* out, void* cuda_stream) {
  TraceRange trace("bmlp_predict");
  return predict_impl(h, x, n, out, cuda_stream, false);
}

int bmlp_predict_layers(bmlp_t* h, const uint64_t* x, int64_t n, int32_t* out, void* cuda_stream) {
  TraceRange trace("bmlp_predict_layers");
  return predict_impl(h, x, n, out, cuda_stream, true);
}

int bmlp_layer_errors(bmlp_t* h, int64_t* errs_out, int32_t reset) {
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (!errs_out) return fail(h, BMLP_EINVAL, "errs_out is NULL");
  CK(h, cudaDeviceSynchronize());
  unsigned long long v[BMLP_MAX_LAYERS];
  CK(h, cudaMemcpy(v, h->dCtrl->layer_err, sizeof(unsigned long long) * h->L, cudaMemcpyDeviceToHost));
  for (int l = 0; l < h->L; ++l) errs_out[l] = (int64_t)v[l];
  if (reset) {
    CK(h, cudaMemset(h->dCtrl->layer_err, 0, sizeof(unsigned long long) * h->L));
    CK(h, cudaDeviceSynchronize());
  }
  return BMLP_OK;
}

int bmlp_binarize_median(const float* x, int64_t n, int32_t K, uint64_t* out, void* cuda_stream) {
  TraceRange trace("bmlp_binarize_median");
  if (n < 0 || K < 1) return fail(nullptr, BMLP_EINVAL, "bmlp_binarize_median: n < 0 or K < 1");
  if (n == 0) return BMLP_OK;
  if (!x || !out || !is_device_ptr(x) || !is_device_ptr(out))
    return fail(nullptr, BMLP_EINVAL, "bmlp_binarize_median: x and out must be device pointers");
  if ((reinterpret_cast<uintptr_t>(x) & 3) || (reinterpret_cast<uintptr_t>(out) & 7))
    return fail(nullptr, BMLP_EINVAL, "bmlp_binarize_median: misaligned x or out");
  launch_binarize_median(x, n, K, (K + 63) / 64, out, static_cast<cudaStream_t>(cuda_stream));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "k_binarize_median");
  return BMLP_OK;
}

int bmlp_expand_weights(uint64_t seed, int32_t K, int32_t D, uint64_t* E_out, void* cuda_stream) {
  TraceRange trace("bmlp_expand_weights");
  if (K < 1 || D < 1 || D > (1 << 23))
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_weights: K < 1, D < 1 or D > 2^23");
  if (!E_out || !is_device_ptr(E_out))
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_weights: E_out must be a device pointer");
  if (reinterpret_cast<uintptr_t>(E_out) & 7)
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_weights: misaligned E_out");
  launch_expand_weights(seed, K, D, E_out, static_cast<cudaStream_t>(cuda_stream));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "k_expand_weights");
  return BMLP_OK;
}

int bmlp_expand_sign(const uint8_t* x, int64_t n, int32_t D, const uint64_t* E, int32_t K,
                     uint64_t* out, void* cuda_stream) {
  TraceRange trace("bmlp_expand_sign");
  if (n < 0 || K < 1 || D < 1 || D > (1 << 23))
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_sign: n < 0, K < 1, D < 1 or D > 2^23");
  if (n == 0) return BMLP_OK;
  if (!x || !E || !out || !is_device_ptr(x) || !is_device_ptr(E) || !is_device_ptr(out))
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_sign: x, E and out must be device pointers");
  if ((reinterpret_cast<uintptr_t>(E) & 7) || (reinterpret_cast<uintptr_t>(out) & 7))
    return fail(nullptr, BMLP_EINVAL, "bmlp_expand_sign: misaligned E or out");
  launch_expand_sign(x, n, D, E, K, out, static_cast<cudaStream_t>(cuda_stream));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(nullptr, e, "k_expand_sign");
  return BMLP_OK;
}

int bmlp_get_state(const bmlp_t* hc, int32_t layer, int16_t* H_out, uint64_t* W_out, int8_t* P_out,
                   double* p_r_out, int64_t* step_out) {
  bmlp_t* h = const_cast<bmlp_t*>(hc);
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (layer < 1 || layer > h->L) return fail(h, BMLP_EINVAL, "layer must be in 1..%d", h->L);
  CK(h, cudaDeviceSynchronize());
  const DevLayer& D = h->hp.layer[layer - 1];
  if (H_out) {
    // bit-sliced lattice indices -> h = 2u - h_max
    std::vector<uint32_t> planes((size_t)D.Kout * D.ldh);
    CK(h, cudaMemcpy(planes.data(), D.H, sizeof(uint32_t) * planes.size(), cudaMemcpyDeviceToHost));
    const int np = h->hp.nplanes;
    for (int64_t k = 0; k < D.Kout; ++k) {
      const uint32_t* row = planes.data() + (size_t)k * D.ldh;
      int16_t* out = H_out + k * D.Kin;
      for (int i = 0; i < D.Kin; ++i) {
        const uint32_t* grp = row + (size_t)(i >> 5) * np;
        int u = 0;
        for (int p = 0; p < np; ++p) u |= (int)((grp[p] >> (i & 31)) & 1u) << p;
        out[i] = (int16_t)(2 * u - h->h_max);
      }
    }
  }
  if (W_out) CK(h, cudaMemcpy(W_out, D.W, sizeof(uint64_t) * D.Kout * D.nw_in, cudaMemcpyDeviceToHost));
  if (P_out) CK(h, cudaMemcpy(P_out, D.rho, (size_t)D.Kout * h->c, cudaMemcpyDeviceToHost));
  if (p_r_out) *p_r_out = h->p_r;
  if (step_out) {
    unsigned long long t = 0;
    CK(h, cudaMemcpy(&t, &h->dCtrl->t, sizeof(t), cudaMemcpyDeviceToHost));
    *step_out = (int64_t)t;
  }
  return BMLP_OK;
}

int bmlp_set_state(bmlp_t* h, int32_t layer, const int16_t* H_in, double p_r, int64_t step) {
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (layer < 1 || layer > h->L) return fail(h, BMLP_EINVAL, "layer must be in 1..%d", h->L);
  const DevLayer& D = h->hp.layer[layer - 1];
  if (H_in) {
    const int64_t cnt = (int64_t)D.Kout * D.Kin;
    for (int64_t i = 0; i < cnt; ++i) {
      const int v = H_in[i];
      if ((v % 2) == 0 || v > h->h_max || v < -h->h_max)
        return fail(h, BMLP_ESTATE, "hidden weight %lld = %d is not odd within [-h_max, h_max]", (long long)i, v);
    }
  }
  if (step >= 0 && (!(p_r >= 0.0) || !std::isfinite(p_r))) return fail(h, BMLP_ESTATE, "p_r invalid");
  CK(h, cudaDeviceSynchronize());
  if (H_in) {
    // h -> bit-sliced lattice index u = (h + h_max)/2 (padding 0)
    const int np = h->hp.nplanes;
    std::vector<uint32_t> planes((size_t)D.Kout * D.ldh, 0u);
    for (int64_t k = 0; k < D.Kout; ++k) {
      uint32_t* row = planes.data() + (size_t)k * D.ldh;
      const int16_t* in = H_in + k * D.Kin;
      for (int i = 0; i < D.Kin; ++i) {
        const int u = (in[i] + h->h_max) / 2;
        uint32_t* grp = row + (size_t)(i >> 5) * np;
        for (int p = 0; p < np; ++p) grp[p] |= (uint32_t)((u >> p) & 1) << (i & 31);
      }
    }
    CK(h, cudaMemcpy(D.H, planes.data(), sizeof(uint32_t) * planes.size(), cudaMemcpyHostToDevice));
    const int64_t nwt = (int64_t)D.Kout * D.ngrp;
    CK(h, cudaMemset(D.W, 0, sizeof(uint64_t) * D.Kout * D.nw_in));
    k_repack_w<<<(unsigned)((nwt + 255) / 256), 256>>>(D.H, D.W, D.Kin, D.Kout, D.ldh, D.ngrp, np,
                                                       h->h_max);
    CK(h, cudaGetLastError());
    h->launches += 1;
  }
  if (step >= 0) {
    h->p_r = p_r;
    unsigned long long t = (unsigned long long)step;
    CK(h, cudaMemcpy(&h->dCtrl->t, &t, sizeof(t), cudaMemcpyHostToDevice));
    h->t_host = step;
    int rc = upload_thresholds(h, 0);
    if (rc != BMLP_OK) return rc;
  }
  CK(h, cudaMemset(&h->dCtrl->err, 0, sizeof(unsigned long long)));
  h->epoch_n = 0;
  CK(h, cudaDeviceSynchronize());
  return BMLP_OK;
}

int bmlp_get_info(const bmlp_t* h, int32_t* n_layers, int32_t* widths_out, int32_t* classes,
                  int32_t* gamma_out, int32_t* bs, int32_t* fwd_impl) {
  if (!h) return BMLP_EINVAL;
  if (n_layers) *n_layers = h->L;
  if (widths_out) for (int l = 0; l <= h->L; ++l) widths_out[l] = h->K[l];
  if (classes) *classes = h->c;
  if (gamma_out) for (int l = 1; l <= h->L; ++l) gamma_out[l - 1] = h->gamma[l];
  if (bs) *bs = h->bs;
  if (fwd_impl) *fwd_impl = h->fwd_impl;
  return BMLP_OK;
}

int bmlp_layer_forward(bmlp_t* h, int32_t layer, const uint64_t* a_in, int64_t n, uint64_t* a_out,
                       void* cuda_stream) {
  TraceRange trace("bmlp_layer_forward");
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (layer < 1 || layer > h->L) return fail(h, BMLP_EINVAL, "layer must be in 1..%d", h->L);
  if (n < 0) return fail(h, BMLP_EINVAL, "n < 0");
  if (n == 0) return BMLP_OK;
  if (!a_in || !a_out || !is_device_ptr(a_in) || !is_device_ptr(a_out))
    return fail(h, BMLP_EINVAL, "a_in and a_out must be device pointers");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const DevLayer& D = h->hp.layer[layer - 1];
  for (int64_t s0 = 0; s0 < n; s0 += kEvalChunk) {
    const int64_t m = std::min(kEvalChunk, n - s0);
    const uint64_t* in = a_in + s0 * D.nw_in;
    uint64_t* out = a_out + s0 * D.nw_out;
    prof_begin(h, kProfEvalFwd, st);
    if (h->fwd_impl == BMLP_FWD_TCGEN05)
      launch_forward_eval_tc(in, m, D.nw_in, D.W, D.Kout, D.Kin, out, D.nw_out,
                             &h->dCtrl->timeouts, st);
    else
      k_forward_eval<<<eval_forward_grid(m, D.Kout), eval_forward_block(), 0, st>>>(
          in, m, D.nw_in, D.W, D.Kout, D.Kin, out, D.nw_out);
    prof_end(h, st);
    CK(h, cudaGetLastError());
    h->launches += 1;
  }
  return prof_collect(h, st);
}

int bmlp_layer_forward_engine(bmlp_t* h, int32_t layer, int32_t engine, const uint64_t* a_in,
                              int64_t n, uint64_t* a_out, void* cuda_stream) {
  TraceRange trace("bmlp_layer_forward_engine");
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (layer < 1 || layer > h->L) return fail(h, BMLP_EINVAL, "layer must be in 1..%d", h->L);
  if (engine != BMLP_FWD_POPC && engine != BMLP_FWD_TCGEN05 && engine != BMLP_FWD_B1MMA)
    return fail(h, BMLP_EINVAL, "engine %d has no layer kernel", engine);
  if (n < 0) return fail(h, BMLP_EINVAL, "n < 0");
  if (n == 0) return BMLP_OK;
  if (!a_in || !a_out || !is_device_ptr(a_in) || !is_device_ptr(a_out))
    return fail(h, BMLP_EINVAL, "a_in and a_out must be device pointers");
  if (engine == BMLP_FWD_TCGEN05) CK(h, prepare_forward_eval_tc());
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const DevLayer& D = h->hp.layer[layer - 1];
  for (int64_t s0 = 0; s0 < n; s0 += kEvalChunk) {
    const int64_t m = std::min(kEvalChunk, n - s0);
    const uint64_t* in = a_in + s0 * D.nw_in;
    uint64_t* out = a_out + s0 * D.nw_out;
    prof_begin(h, kProfEvalFwd, st);
    if (engine == BMLP_FWD_TCGEN05)
      launch_forward_eval_tc(in, m, D.nw_in, D.W, D.Kout, D.Kin, out, D.nw_out,
                             &h->dCtrl->timeouts, st);
    else if (engine == BMLP_FWD_B1MMA)
      CK(h, launch_forward_b1(in, m, D.nw_in, D.W, D.Kout, D.Kin, out, D.nw_out, st));
    else
      k_forward_eval<<<eval_forward_grid(m, D.Kout), eval_forward_block(), 0, st>>>(
          in, m, D.nw_in, D.W, D.Kout, D.Kin, out, D.nw_out);
    prof_end(h, st);
    CK(h, cudaGetLastError());
    h->launches += 1;
  }
  return prof_collect(h, st);
}

int bmlp_debug_wait_probe(bmlp_t* h, int32_t arrive, double seconds) {
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (!(seconds > 0.0) || seconds > 10.0) return fail(h, BMLP_EINVAL, "seconds must be in (0, 10]");
  int khz = 0;
  CK(h, cudaDeviceGetAttribute(&khz, cudaDevAttrClockRate, h->device));
  const unsigned long long limit = (unsigned long long)(seconds * 1e3 * (double)khz);
  launch_wait_probe(&h->dCtrl->timeouts, arrive > 0 ? 1 : 0, limit, 0);
  CK(h, cudaGetLastError());
  CK(h, cudaDeviceSynchronize());
  if (arrive < 0) return BMLP_OK;  // the expiry stays pending for the next synchronising call
  uint32_t t = 0;
  CK(h, cudaMemcpy(&t, &h->dCtrl->timeouts, sizeof(t), cudaMemcpyDeviceToHost));
  if (t != 0) {
    CK(h, cudaMemset(&h->dCtrl->timeouts, 0, sizeof(uint32_t)));
    return fail(h, BMLP_ETIMEOUT, "a bounded device-side wait expired");
  }
  return BMLP_OK;
}

int bmlp_debug_fail_alloc(int64_t nth) {
  if (nth < 0) return fail(nullptr, BMLP_EINVAL, "nth must be >= 0");
  g_fail_at.store(0);
  g_alloc_seq.store(0);
  g_fail_at.store(nth);
  return BMLP_OK;
}

int bmlp_debug_alloc_stats(int64_t* live_allocs, int64_t* live_bytes) {
  if (live_allocs) *live_allocs = g_live_allocs.load();
  if (live_bytes) *live_bytes = g_live_bytes.load();
  return BMLP_OK;
}

int bmlp_engine_peak(int32_t engine, int64_t iters, double* bitpairs_per_s, double* ms_out) {
  TraceRange trace("bmlp_engine_peak");
  g_create_error.clear();
  if (!bitpairs_per_s) return fail(nullptr, BMLP_EINVAL, "bitpairs_per_s is NULL");
  if (engine != BMLP_FWD_POPC && engine != BMLP_FWD_TCGEN05 && engine != BMLP_FWD_B1MMA &&
      engine != BMLP_FWD_S8MMA)
    return fail(nullptr, BMLP_EINVAL, "unknown engine %d", engine);
  if (iters < 1 || iters > (int64_t)1 << 31) return fail(nullptr, BMLP_EINVAL, "iters out of range");
  int dev = 0, sms = 0;
  CK(nullptr, cudaGetDevice(&dev));
  CK(nullptr, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  int* sink = nullptr;
  unsigned int* tmo = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  int rc = BMLP_OK;
  double bp = 0.0;
  float ms = 0.f;
  auto step = [&](cudaError_t x, const char* what) {
    if (rc == BMLP_OK && x != cudaSuccess) rc = cuda_fail(nullptr, x, what);
  };
  step(cudaMalloc(&sink, sizeof(int) * 8 * (size_t)sms), "cudaMalloc");
  step(cudaMalloc(&tmo, sizeof(unsigned int)), "cudaMalloc");
  if (rc == BMLP_OK) step(cudaMemset(tmo, 0, sizeof(unsigned int)), "cudaMemset");
  if (rc == BMLP_OK) step(cudaEventCreate(&e0), "cudaEventCreate");
  if (rc == BMLP_OK) step(cudaEventCreate(&e1), "cudaEventCreate");
  // one untimed launch (clocks up, first-launch costs paid), then the timed one
  if (rc == BMLP_OK)
    step(launch_engine_peak(engine, std::max<int64_t>(1, iters / 4), sms, sink, tmo, 0, &bp), "peak kernel");
  if (rc == BMLP_OK) step(cudaEventRecord(e0, 0), "cudaEventRecord");
  if (rc == BMLP_OK) step(launch_engine_peak(engine, iters, sms, sink, tmo, 0, &bp), "peak kernel");
  if (rc == BMLP_OK) step(cudaEventRecord(e1, 0), "cudaEventRecord");
  if (rc == BMLP_OK) step(cudaEventSynchronize(e1), "peak kernel");
  if (rc == BMLP_OK) step(cudaEventElapsedTime(&ms, e0, e1), "cudaEventElapsedTime");
  unsigned int t = 0;
  if (rc == BMLP_OK) step(cudaMemcpy(&t, tmo, sizeof(t), cudaMemcpyDeviceToHost), "cudaMemcpy");
  if (rc == BMLP_OK && t != 0) rc = fail(nullptr, BMLP_ETIMEOUT, "a bounded device-side wait expired");
  if (rc == BMLP_OK) {
    *bitpairs_per_s = bp / ((double)ms * 1e-3);
    if (ms_out) *ms_out = ms;
  }
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (sink) cudaFree(sink);
  if (tmo) cudaFree(tmo);
  return rc;
}

int bmlp_debug_last_step(const bmlp_t* hc, int32_t layer, int16_t* Z, uint64_t* A, uint8_t* mark,
                         int16_t* sel) {
  bmlp_t* h = const_cast<bmlp_t*>(hc);
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  if (layer < 1 || layer > h->L) return fail(h, BMLP_EINVAL, "layer must be in 1..%d", h->L);
  CK(h, cudaDeviceSynchronize());
  const DevLayer& D = h->hp.layer[layer - 1];
  if (Z) CK(h, cudaMemcpy(Z, D.Z, sizeof(int16_t) * h->bs * D.Kout, cudaMemcpyDeviceToHost));
  if (A) CK(h, cudaMemcpy(A, D.A, sizeof(uint64_t) * h->bs * D.nw_out, cudaMemcpyDeviceToHost));
  if (mark) CK(h, cudaMemcpy(mark, D.mark, (size_t)h->bs, cudaMemcpyDeviceToHost));
  if (sel) {
    // device layout [G][bs] -> the documented [bs][G]
    std::vector<int16_t> t((size_t)h->bs * D.G);
    CK(h, cudaMemcpy(t.data(), D.sel, sizeof(int16_t) * t.size(), cudaMemcpyDeviceToHost));
    for (int g = 0; g < D.G; ++g)
      for (int m = 0; m < h->bs; ++m) sel[(size_t)m * D.G + g] = t[(size_t)g * h->bs + m];
  }
  return BMLP_OK;
}

int bmlp_set_profiling(bmlp_t* h, int32_t every) {
  if (!h || every < 0) return BMLP_EINVAL;
  h->profEvery = every;
  h->profiling = every > 0;
  return BMLP_OK;
}

int bmlp_get_profile(const bmlp_t* h, int32_t kind, int64_t* launches, double* total_ms) {
  if (!h || kind < 0 || kind >= kProfKinds) return BMLP_EINVAL;
  if (launches) *launches = h->profN[kind];
  if (total_ms) *total_ms = h->profMs[kind];
  return BMLP_OK;
}

int bmlp_reset_profile(bmlp_t* h) {
  if (!h) return BMLP_EINVAL;
  for (int i = 0; i < kProfKinds; ++i) { h->profN[i] = 0; h->profMs[i] = 0.0; }
  return BMLP_OK;
}

int64_t bmlp_launch_count(const bmlp_t* h) { return h ? h->launches : -1; }

int bmlp_update_stats(bmlp_t* h, int64_t* rows_out, int64_t* streamed_out, int64_t* bytes_out,
                      int32_t reset) {
  if (!h) return BMLP_EINVAL;
  h->err.clear();
  unsigned long long v[3];
  CK(h, cudaDeviceSynchronize());
  CK(h, cudaMemcpy(v, &h->dCtrl->upd_rows, sizeof(v), cudaMemcpyDeviceToHost));
  if (rows_out) *rows_out = (int64_t)v[0];
  if (streamed_out) *streamed_out = (int64_t)v[1];
  if (bytes_out) *bytes_out = (int64_t)v[2];
  if (reset) CK(h, cudaMemset(&h->dCtrl->upd_rows, 0, sizeof(v)));
  return BMLP_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Internal accessors for bmlp_noalloc.cu (not part of the C-ABI).
int bmlp_internal_eval_view(const bmlp_t* h, const bk::StepParams** params, int* nwmax) {
  if (!h) return BMLP_EINVAL;
  *params = &h->hp;
  int m = 0;
  for (int l = 1; l <= h->L; ++l) m = std::max(m, (h->K[l] + 63) / 64);
  *nwmax = m;
  return BMLP_OK;
}

int bmlp_internal_fail(bmlp_t* h, int code, const char* msg) { return fail(h, code, "%s", msg); }

void bmlp_internal_clear_error(bmlp_t* h) {
  if (h) h->err.clear();
}

void bmlp_internal_count_launches(bmlp_t* h, int64_t n) { h->launches += n; }
