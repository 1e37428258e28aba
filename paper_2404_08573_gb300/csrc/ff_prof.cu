// Launch accounting and optional per-kernel timing.
//
// Every kernel launch libff makes is counted.  While timing is enabled
// (ff_profile_enable(1)), each launch is also bracketed by two CUDA events
// recorded on the stream the kernel is launched on, and tagged with the
// kernel kind and its algorithmic work (FLOPs for the GEMMs, bytes that the
// algorithm must move for the bandwidth-bound kernels).  ff_profile_read
// waits for the recorded events and returns per-kind totals.
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <mutex>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "ff_prof.h"

namespace ff {
namespace {

const char* const kNames[K_NUM] = {"overlay",     "row_scale",    "fwd_gemm_tc",   "fwd_gemm_simt",
                                   "finalize",    "grad_prep",   "wgrad_gemm_tc", "wgrad_gemm_simt",
                                   "adam",        "init_weights", "to_bf16",       "label_columns",
                                   "store_gemm_tc", "store_gemm_simt", "expand",   "argmax",
                                   "head_logits", "head_wgrad",   "head_adam",
                                   "epoch_gemm_tc"};

struct Rec {
  int kind;
  double work;
  cudaEvent_t a, b;
  cudaStream_t st;
};

std::mutex mu;
bool enabled = false;
std::vector<Rec> recs;
std::vector<cudaEvent_t> pool;
std::atomic<unsigned long long> launches{0};

cudaEvent_t take() {
  if (!pool.empty()) {
    cudaEvent_t e = pool.back();
    pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

}  // namespace

long long launch_fail_at() {
  static const long long v = [] {
    const char* e = std::getenv("FF_FAULT_LAUNCH_FAIL_AT");
    return e ? std::atoll(e) : 0ll;
  }();
  return v;
}

ProfScope::ProfScope(KernelKind k, double work, cudaStream_t st) : kind_(k), work_(work), st_(st) {
  const unsigned long long nth = launches.fetch_add(1, std::memory_order_relaxed) + 1;
  const long long f = launch_fail_at();
  if (f > 0 && nth == (unsigned long long)f) {
    injected_ = true;
    return;
  }
  std::lock_guard<std::mutex> g(mu);
  if (!enabled) return;
  a_ = take();
  b_ = take();
  if (a_ && b_) {
    cudaEventRecord(a_, st_);
  } else {
    if (a_) pool.push_back(a_);
    if (b_) pool.push_back(b_);
    a_ = b_ = nullptr;
  }
}

ProfScope::~ProfScope() {
  if (!a_) return;
  std::lock_guard<std::mutex> g(mu);
  cudaEventRecord(b_, st_);
  recs.push_back(Rec{kind_, work_, a_, b_, st_});
}

ff_status injected_launch_failure(const char* what) {
  if (std::getenv("FF_DEBUG")) std::fprintf(stderr, "libff: %s: injected launch failure\n", what);
  return FF_ERR_CUDA;
}

NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

}  // namespace ff

using namespace ff;

extern "C" {

ff_status ff_profile_enable(int on) {
  std::lock_guard<std::mutex> g(mu);
  if (on) {
    for (auto& r : recs) {
      pool.push_back(r.a);
      pool.push_back(r.b);
    }
    recs.clear();
  }
  enabled = on != 0;
  return FF_OK;
}

int ff_profile_read(int capacity, const char** names, long long* count, double* ms, double* work) {
  std::lock_guard<std::mutex> g(mu);
  long long c[K_NUM] = {0};
  double t[K_NUM] = {0}, w[K_NUM] = {0};
  for (auto& r : recs) {
    if (cudaEventSynchronize(r.b) != cudaSuccess) return -1;
    float e = 0.f;
    if (cudaEventElapsedTime(&e, r.a, r.b) != cudaSuccess) return -1;
    c[r.kind] += 1;
    t[r.kind] += e;
    w[r.kind] += r.work;
  }
  int n = 0;
  for (int k = 0; k < K_NUM && n < capacity; ++k) {
    if (!c[k]) continue;
    if (names) names[n] = kNames[k];
    if (count) count[n] = c[k];
    if (ms) ms[n] = t[k];
    if (work) work[n] = w[k];
    ++n;
  }
  return n;
}

unsigned long long ff_kernel_launches(void) { return launches.load(std::memory_order_relaxed); }

int ff_profile_timeline(int capacity, int* kind, long long* stream_id, double* start_ms, double* end_ms) {
  std::lock_guard<std::mutex> g(mu);
  if (recs.empty()) return 0;
  if (cudaEventSynchronize(recs.back().b) != cudaSuccess) return -1;
  // the earliest start among the records is the time origin
  size_t first = 0;
  for (size_t i = 1; i < recs.size(); ++i) {
    float d = 0.f;
    if (cudaEventElapsedTime(&d, recs[first].a, recs[i].a) != cudaSuccess) return -1;
    if (d < 0) first = i;
  }
  int n = 0;
  for (size_t i = 0; i < recs.size() && n < capacity; ++i, ++n) {
    float t0 = 0.f, t1 = 0.f;
    if (cudaEventElapsedTime(&t0, recs[first].a, recs[i].a) != cudaSuccess) return -1;
    if (cudaEventElapsedTime(&t1, recs[first].a, recs[i].b) != cudaSuccess) return -1;
    if (kind) kind[n] = recs[i].kind;
    if (stream_id) stream_id[n] = (long long)reinterpret_cast<uintptr_t>(recs[i].st);
    if (start_ms) start_ms[n] = t0;
    if (end_ms) end_ms[n] = t1;
  }
  return n;
}

const char* ff_profile_kind_name(int kind) { return (kind >= 0 && kind < K_NUM) ? kNames[kind] : "unknown"; }

}  // extern "C"
