// A net of FF layers trained concurrently on one GPU, one CUDA stream per
// layer: the single-GPU analogue of Single-Layer PFF (§4.1, Algorithm 1),
// where node i trains L_i on the output of L_{i-1} while node i-1 already
// trains further.  Here the hand-off is per batch through ring buffers of
// `depth` activation slots per layer boundary:
//   layer k, batch t: waits ready[k-1][t % depth] (layer k-1's forward of
//   batch t is written) and, before overwriting its own output slot,
//   consumed[k][t % depth] (layer k+1 has finished batch t - depth).
// Each layer's own steps stay in order on its stream, so every kernel sees
// exactly the inputs it would see in a one-stream run: results are bitwise
// identical to the sequential schedule.
//
// A Performance-Optimized net (§4, ff_net_create_po) runs the same way with
// ff_po_train_step per layer and block: batch t's labels, which every layer
// reads, are copied into a ring slot by layer 1's stream and the slot is
// reused only after the last layer has finished with it.
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "ff_api_internal.h"
#include "ff_net_internal.h"
#include "ff_prof.h"


namespace {

void release(ff_net* n) {
  if (!n) return;
  for (auto st : n->streams)
    if (st) cudaStreamSynchronize(st);
  // the layers outlive the net: they must not keep a stream that is about to go away
  for (auto* l : n->layers)
    for (auto st : n->streams)
      if (l && st && l->last_stream == st) l->last_stream = nullptr;
  for (auto* b : n->blocks)
    for (auto st : n->streams)
      if (b && st) ff::head_forget_stream(b, st);
  for (auto e : n->lab_done)
    if (e) cudaEventDestroy(e);
  for (auto& v : n->ready)
    for (auto e : v)
      if (e) cudaEventDestroy(e);
  for (auto& v : n->consumed)
    for (auto e : v)
      if (e) cudaEventDestroy(e);
  for (auto e : n->tail)
    if (e) cudaEventDestroy(e);
  if (n->ev_x_in) cudaEventDestroy(n->ev_x_in);
  if (n->ev_x_done) cudaEventDestroy(n->ev_x_done);
  for (auto st : n->streams)
    if (st) cudaStreamDestroy(st);
  ff::epoch_plan_free(n->epoch);
  ff::dev_free(n->mem);
  delete n;
}

}  // namespace

extern "C" {

}  // extern "C"

namespace {

// Shared by ff_net_create (rows = 2 * max_B pairs) and ff_net_create_po
// (rows = max_rows samples, with blocks).
ff_status create_net(ff_layer* const* layers, ff_head* const* blocks, int n_layers, int rows, int depth,
                     ff_net** out) {
  if (!out) return FF_ERR_INVALID_ARG;
  *out = nullptr;
  if (!layers || n_layers < 1 || rows < 1 || depth < 1 || depth > 64) return FF_ERR_INVALID_ARG;
  for (int k = 0; k < n_layers; ++k) {
    if (!layers[k]) return FF_ERR_INVALID_ARG;
    if (k > 0 && (layers[k]->K != layers[k - 1]->N || layers[k]->is_bf16 != layers[0]->is_bf16)) return FF_ERR_INVALID_ARG;
    for (int j = 0; j < k; ++j)
      if (layers[j] == layers[k]) return FF_ERR_INVALID_ARG;
  }
  if (layers[0]->K < 10) return FF_ERR_INVALID_ARG;
  ff_net* n = new (std::nothrow) ff_net();
  if (!n) return FF_ERR_OOM;
  n->layers.assign(layers, layers + n_layers);
  n->L = n_layers;
  n->max_B = rows / 2;
  n->max_rows = rows;
  n->depth = depth;
  n->po = blocks != nullptr;
  if (n->po) n->blocks.assign(blocks, blocks + n_layers);
  const size_t M = (size_t)rows;
  const size_t es = layers[0]->is_bf16 ? 2 : 4;
  size_t total = 0;
  for (int k = 0; k + 1 < n_layers; ++k)
    total += (size_t)depth * (((M * layers[k]->ldN * es + 255) & ~(size_t)255) + ((M * 4 + 255) & ~(size_t)255));
  if (n->po) total += (size_t)depth * ((M * 4 + 255) & ~(size_t)255);
  ff_status s = FF_OK;
  if (total) s = ff::cuda_status(ff::dev_alloc(&n->mem, total), "net activation buffers");
  if (s != FF_OK) {
    release(n);
    return s;
  }
  char* p = static_cast<char*>(n->mem);
  n->hbuf.resize(n_layers > 1 ? n_layers - 1 : 0);
  n->sbuf.resize(n->hbuf.size());
  n->ready.resize(n->hbuf.size());
  n->consumed.resize(n->hbuf.size());
  for (int k = 0; k + 1 < n_layers; ++k) {
    for (int d = 0; d < depth; ++d) {
      n->hbuf[k].push_back(p);
      p += (M * layers[k]->ldN * es + 255) & ~(size_t)255;
      n->sbuf[k].push_back(reinterpret_cast<float*>(p));
      p += (M * 4 + 255) & ~(size_t)255;
      cudaEvent_t e1 = nullptr, e2 = nullptr;
      cudaError_t e = cudaEventCreateWithFlags(&e1, cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&e2, cudaEventDisableTiming);
      n->ready[k].push_back(e1);
      n->consumed[k].push_back(e2);
      if (e != cudaSuccess) {
        release(n);
        return ff::cuda_status(e, "net events");
      }
    }
  }
  for (int d = 0; n->po && d < depth; ++d) {
    n->lab.push_back(reinterpret_cast<int*>(p));
    p += (M * 4 + 255) & ~(size_t)255;
    cudaEvent_t ev = nullptr;
    cudaError_t e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    n->lab_done.push_back(ev);
    if (e != cudaSuccess) {
      release(n);
      return ff::cuda_status(e, "net events");
    }
  }
  for (int k = 0; k < n_layers; ++k) {
    cudaStream_t st = nullptr;
    cudaEvent_t ev = nullptr;
    cudaError_t e = cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking);
    n->streams.push_back(st);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    n->tail.push_back(ev);
    if (e != cudaSuccess) {
      release(n);
      return ff::cuda_status(e, "net streams");
    }
  }
  cudaError_t e = cudaEventCreateWithFlags(&n->ev_x_in, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&n->ev_x_done, cudaEventDisableTiming);
  if (e != cudaSuccess) {
    release(n);
    return ff::cuda_status(e, "net events");
  }
  *out = n;
  return FF_OK;
}

}  // namespace

namespace ff {

// One batch through every layer; images_once: x holds one image per pair.
ff_status net_train_step(ff_net* n, const float* x, const int* labels, int B, float* loss, void* stream,
                                bool images_once) {
  if (!n || !x || !labels || B < 0 || B > n->max_B || n->po) return FF_ERR_INVALID_ARG;
  if (B == 0) return FF_OK;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int slot = (int)(n->step % n->depth);
  ff_status s = ff::cuda_status(cudaEventRecord(n->ev_x_in, cs), "record input event");
  if (s != FF_OK) return s;
  for (int k = 0; k < n->L; ++k) {
    cudaStream_t st = n->streams[k];
    cudaError_t e = cudaStreamWaitEvent(st, k == 0 ? n->ev_x_in : n->ready[k - 1][slot], 0);
    // Before overwriting its output slot, layer k waits until layer k+1 has
    // read what batch t - depth left there.  Within `depth` steps after an
    // ff_net_sync that read is already ordered before this point (every
    // stream joined the caller's stream, which this step's input event
    // follows), so no wait is issued: a synced run of steps is self-contained
    // and can be captured in a CUDA graph.
    if (e == cudaSuccess && k + 1 < n->L && n->since_sync >= n->depth)
      e = cudaStreamWaitEvent(st, n->consumed[k][slot], 0);
    s = ff::cuda_status(e, "stream wait");
    if (s != FF_OK) return s;
    const void* xin = k == 0 ? static_cast<const void*>(x) : n->hbuf[k - 1][slot];
    const float* scale = k == 0 ? nullptr : n->sbuf[k - 1][slot];
    void* hout = k + 1 < n->L ? n->hbuf[k][slot] : nullptr;
    float* sn = k + 1 < n->L ? n->sbuf[k][slot] : nullptr;
    s = ff::train_step_impl(n->layers[k], xin, k == 0 ? labels : nullptr, scale, B, hout, sn, nullptr,
                            loss ? loss + k : nullptr, st, k == 0 ? n->ev_x_done : nullptr,
                            k + 1 < n->L ? n->ready[k][slot] : nullptr, images_once && k == 0);
    if (s != FF_OK) return s;
    if (k > 0) {
      s = ff::cuda_status(cudaEventRecord(n->consumed[k - 1][slot], st), "record consumed event");
      if (s != FF_OK) return s;
    }
  }
  s = ff::cuda_status(cudaStreamWaitEvent(cs, n->ev_x_done, 0), "input hand-back");
  if (s != FF_OK) return s;
  ++n->step;
  ++n->since_sync;
  return FF_OK;
}

}  // namespace ff

extern "C" {

ff_status ff_net_create(ff_layer* const* layers, int n_layers, int max_B, int depth, ff_net** out) {
  if (max_B < 1 || max_B > (1 << 29)) {
    if (out) *out = nullptr;
    return FF_ERR_INVALID_ARG;
  }
  return create_net(layers, nullptr, n_layers, 2 * max_B, depth, out);
}

ff_status ff_net_create_po(ff_layer* const* layers, ff_head* const* blocks, int n_layers, int max_rows, int depth,
                           ff_net** out) {
  if (!blocks || !layers || n_layers < 1) {
    if (out) *out = nullptr;
    return FF_ERR_INVALID_ARG;
  }
  for (int k = 0; k < n_layers; ++k)
    if (!blocks[k] || !layers[k] || ff::head_features(blocks[k]) != layers[k]->N) {
      if (out) *out = nullptr;
      return FF_ERR_INVALID_ARG;
    }
  return create_net(layers, blocks, n_layers, max_rows, depth, out);
}

ff_status ff_net_destroy(ff_net* n) {
  release(n);
  return FF_OK;
}

ff_status ff_net_po_train_step(ff_net* n, const float* x, const int* labels, int rows, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_net_po_train_step");
  if (!n || !x || !labels || rows < 0 || rows > n->max_rows || !n->po) return FF_ERR_INVALID_ARG;
  if (rows == 0) return FF_OK;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int slot = (int)(n->step % n->depth);
  const bool wait_reuse = n->since_sync >= n->depth;
  ff_status s = ff::cuda_status(cudaEventRecord(n->ev_x_in, cs), "record input event");
  if (s != FF_OK) return s;
  int* lab = n->lab[slot];
  for (int k = 0; k < n->L; ++k) {
    cudaStream_t st = n->streams[k];
    cudaError_t e = cudaStreamWaitEvent(st, k == 0 ? n->ev_x_in : n->ready[k - 1][slot], 0);
    if (e == cudaSuccess && k + 1 < n->L && wait_reuse) e = cudaStreamWaitEvent(st, n->consumed[k][slot], 0);
    if (e == cudaSuccess && k == 0) {
      // this batch's labels into the ring slot, once the last layer is done with it
      if (wait_reuse) e = cudaStreamWaitEvent(st, n->lab_done[slot], 0);
      if (e == cudaSuccess) e = cudaMemcpyAsync(lab, labels, (size_t)rows * 4, cudaMemcpyDeviceToDevice, st);
    }
    s = ff::cuda_status(e, "stream wait");
    if (s != FF_OK) return s;
    const void* xin = k == 0 ? static_cast<const void*>(x) : n->hbuf[k - 1][slot];
    const float* scale = k == 0 ? nullptr : n->sbuf[k - 1][slot];
    void* hout = k + 1 < n->L ? n->hbuf[k][slot] : nullptr;
    float* sn = k + 1 < n->L ? n->sbuf[k][slot] : nullptr;
    s = ff_po_train_step(n->layers[k], n->blocks[k], xin, k == 0 ? 1 : 0, scale, lab, rows, hout, sn,
                         loss ? loss + k : nullptr, st);
    if (s != FF_OK) return s;
    if (k + 1 < n->L) s = ff::cuda_status(cudaEventRecord(n->ready[k][slot], st), "record ready event");
    if (s == FF_OK && k > 0) s = ff::cuda_status(cudaEventRecord(n->consumed[k - 1][slot], st), "record consumed event");
    if (s == FF_OK && k == 0) s = ff::cuda_status(cudaEventRecord(n->ev_x_done, st), "record input event");
    if (s == FF_OK && k + 1 == n->L) s = ff::cuda_status(cudaEventRecord(n->lab_done[slot], st), "record label event");
    if (s != FF_OK) return s;
  }
  s = ff::cuda_status(cudaStreamWaitEvent(cs, n->ev_x_done, 0), "input hand-back");
  if (s != FF_OK) return s;
  ++n->step;
  ++n->since_sync;
  return FF_OK;
}

ff_status ff_net_train_step(ff_net* n, const float* x, const int* labels, int B, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_net_train_step");
  return ff::net_train_step(n, x, labels, B, loss, stream, false);
}

ff_status ff_net_train_step_images(ff_net* n, const float* x, const int* labels, int B, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_net_train_step_images");
  return ff::net_train_step(n, x, labels, B, loss, stream, true);
}

ff_status ff_net_sync(ff_net* n, void* stream) {
  if (!n) return FF_ERR_INVALID_ARG;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  for (int k = 0; k < n->L; ++k) {
    cudaError_t e = cudaEventRecord(n->tail[k], n->streams[k]);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, n->tail[k], 0);
    ff_status s = ff::cuda_status(e, "net sync");
    if (s != FF_OK) return s;
  }
  n->since_sync = 0;
  return FF_OK;
}

ff_status ff_net_wait(ff_net* n, unsigned timeout_ms) {
  if (!n) return FF_ERR_INVALID_ARG;
  for (int k = 0; k < n->L; ++k) {
    ff_status s = ff::cuda_status(cudaEventRecord(n->tail[k], n->streams[k]), "net wait");
    if (s != FF_OK) return s;
  }
  ff_status s = ff::wait_events(n->tail.data(), n->L, timeout_ms);
  if (s == FF_OK) n->since_sync = 0;  // everything enqueued so far has finished
  return s;
}

}  // extern "C"
