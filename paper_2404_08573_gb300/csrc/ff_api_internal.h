// Host-side helpers shared by ff_api.cu and ff_net.cu.
#pragma once

#include "ff_internal.cuh"
#include "ff_prof.h"

namespace ff {

ff_status cuda_status(cudaError_t e, const char* what);
cudaError_t dev_alloc(void** p, size_t bytes);
void dev_free(void* p);

// Host-side bounded wait: polls the events until all have completed
// (FF_OK) or timeout_ms has passed (FF_ERR_TIMEOUT); a failed event query is
// reported as its CUDA status.
ff_status wait_events(const cudaEvent_t* ev, int n, unsigned timeout_ms);

// Softmax heads (ff_head.cu): the feature count, and dropping a stream that
// is about to be destroyed from the head's bookkeeping.
int head_features(const ff_head* h);
void head_forget_stream(ff_head* h, cudaStream_t st);

// Grows the layer's workspace to at least `rows` rows (waits for the layer's
// last stream before replacing it).
ff_status ensure_capacity(ff_layer* L, int rows);

// One layer-local train step (see ff_layer_train_step).  ev_input_read, if
// not null, is recorded once the raw input x has been consumed (after the
// overlay; only meaningful when labels are given); ev_forward_done, if not
// null, once the activity, goodness and next-layer scale are written.
// images_once (with labels): x holds B images, one per pair, read for both
// the positive row i and the negative row B + i.
ff_status train_step_impl(ff_layer* L, const void* x, const int* labels, const float* row_scale, int B,
                          void* h_out, float* next_scale, float* goodness, float* loss, cudaStream_t st,
                          cudaEvent_t ev_input_read, cudaEvent_t ev_forward_done, bool images_once = false);

}  // namespace ff

#define FF_TRY(call, what)                                 \
  do {                                                     \
    ff_status s_ = ::ff::cuda_status((call), (what));      \
    if (s_ != FF_OK) return s_;                            \
  } while (0)

// A kernel launch: counted, and timed on its stream while profiling is on.
#define FF_LAUNCH(kind, work, st, call, what)                          \
  do {                                                                 \
    ff_status s_;                                                      \
    {                                                                  \
      ::ff::ProfScope p_((kind), (double)(work), (st));                \
      s_ = p_.injected_failure() ? ::ff::injected_launch_failure(what) \
                                 : ::ff::cuda_status((call), (what));  \
    }                                                                  \
    if (s_ != FF_OK) return s_;                                        \
  } while (0)
