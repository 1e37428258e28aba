// Launch accounting and optional per-kernel event timing (see ff_prof.cu).
#pragma once

#include "ff_internal.cuh"

namespace ff {

enum KernelKind {
  K_OVERLAY, K_ROW_SCALE, K_FWD_TC, K_FWD_SIMT, K_FINALIZE, K_GRAD_PREP, K_WGRAD_TC, K_WGRAD_SIMT,
  K_ADAM, K_INIT, K_TO_BF16, K_LABEL_COLS, K_STORE_TC, K_STORE_SIMT, K_EXPAND, K_ARGMAX,
  K_HEAD_LOGITS, K_HEAD_FINISH, K_HEAD_WGRAD, K_HEAD_ADAM, K_NUM
};

// Counts one launch; when timing is enabled records an event on `st` now and
// another when the scope ends (place the launch inside the scope).
class ProfScope {
 public:
  ProfScope(KernelKind k, double work, cudaStream_t st);
  ~ProfScope();
  ProfScope(const ProfScope&) = delete;
  ProfScope& operator=(const ProfScope&) = delete;

 private:
  int kind_;
  double work_;
  cudaStream_t st_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
};

}  // namespace ff
