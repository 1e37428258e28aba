// Launch accounting and optional per-kernel event timing (see ff_prof.cu).
#pragma once

#include "ff_internal.cuh"

namespace ff {

enum KernelKind {
  K_OVERLAY, K_ROW_SCALE, K_FWD_TC, K_FWD_SIMT, K_FINALIZE, K_GRAD_PREP, K_WGRAD_TC, K_WGRAD_SIMT,
  K_ADAM, K_INIT, K_TO_BF16, K_LABEL_COLS, K_STORE_TC, K_STORE_SIMT, K_EXPAND, K_ARGMAX,
  K_HEAD_LOGITS, K_HEAD_WGRAD, K_HEAD_ADAM, K_EPOCH, K_NUM
};

// Counts one launch; when timing is enabled records an event on `st` now and
// another when the scope ends (place the launch inside the scope).
class ProfScope {
 public:
  ProfScope(KernelKind k, double work, cudaStream_t st);
  ~ProfScope();
  // Host-side fault injection: with FF_FAULT_LAUNCH_FAIL_AT=n in the
  // environment, the n-th launch of the process (1-based) is not made and
  // its call reports a launch failure.
  bool injected_failure() const { return injected_; }
  ProfScope(const ProfScope&) = delete;
  ProfScope& operator=(const ProfScope&) = delete;

 private:
  int kind_;
  double work_;
  cudaStream_t st_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
  bool injected_ = false;
};

// The status a call returns for an injected launch failure.
ff_status injected_launch_failure(const char* what);

// NVTX range over the scope (shown by profilers that record NVTX; free
// otherwise).
class NvtxRange {
 public:
  explicit NvtxRange(const char* name);
  ~NvtxRange();
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

}  // namespace ff
