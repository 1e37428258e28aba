// The net object behind the opaque ff_net handle (ff_net.cu), shared with
// the persistent train-epoch path (ff_epoch.cu).
#pragma once

#include <vector>

#include "ff_api_internal.h"

namespace ff {
struct EpochPlan;
void epoch_plan_free(EpochPlan* p);
// One batch through every layer of a (non-PO) net on its layer streams
// (ff_net_train_step; images_once: x holds one image per pair).
ff_status net_train_step(ff_net* n, const float* x, const int* labels, int B, float* loss, void* stream,
                         bool images_once);
}  // namespace ff

struct ff_net {
  std::vector<ff_layer*> layers;
  int L = 0, max_B = 0, depth = 0;
  std::vector<cudaStream_t> streams;
  std::vector<std::vector<void*>> hbuf;
  std::vector<std::vector<float*>> sbuf;
  std::vector<std::vector<cudaEvent_t>> ready, consumed;
  std::vector<cudaEvent_t> tail;
  cudaEvent_t ev_x_in = nullptr, ev_x_done = nullptr;
  long long step = 0;
  long long since_sync = 0;  // steps enqueued since the last ff_net_sync
  void* mem = nullptr;
  // Performance-Optimized nets: one softmax block per layer, label ring
  bool po = false;
  int max_rows = 0;
  std::vector<ff_head*> blocks;
  std::vector<int*> lab;
  std::vector<cudaEvent_t> lab_done;
  // the persistent train-epoch plan (ff_net_train_epoch), built on first use
  ff::EpochPlan* epoch = nullptr;
  bool epoch_trace = false;  // record per-task times in the epoch kernel (ff_net_epoch_trace)
};

