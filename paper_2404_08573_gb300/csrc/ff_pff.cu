// Chapter schedule of the pipelined FF algorithms (§4) on one GPU.
//
// The E training epochs are cut into S chapters of C = E/S epochs.  In
// chapter c, layer i trains C epochs over the output of layer i-1 as that
// layer stands after its own chapter c (layer 1: the raw pairs overlaid with
// the chapter's labels), then publishes its output -- a forward pass of the
// whole training set with the updated weights -- for layer i+1.  So layer i's
// chapter c depends on layer i-1's chapter c and on its own chapter c-1, and
// nothing else: a wavefront over (layer, chapter).
//
//   Single-Layer PFF (Algorithm 1): one CUDA stream per layer, as one node
//     per layer;
//   All-Layers PFF (Algorithm 2): `nodes` streams take the chapters in turn,
//     each training every layer of its chapter.
//
// Both run the same dependency graph with the same kernels, so they give the
// same weights bit for bit; they differ in which work can overlap.  A layer's
// published output lives in HBM (two chapter slots per layer), where the
// paper's nodes send layers over the network instead.  Enqueueing follows the
// wavefront t = c + i, and every cross-stream dependency is an event.
#include <cmath>
#include <new>
#include <vector>

#include "ff_api_internal.h"
#include "ff_prof.h"
#include "ff_internal.cuh"

struct ff_pff {
  ff_pff_config cfg;
  std::vector<ff_layer*> layers;
  std::vector<float> lr0;          // each layer's configured learning rate
  std::vector<cudaStream_t> streams;
  // published outputs of layers 0..L-2: two chapter slots each
  std::vector<void*> pub[2];
  std::vector<float*> pubs[2];
  void* pub_mem = nullptr;
  // ev_pub[i][slot]: layer i's output of the chapter in `slot` is written;
  // ev_read[i][slot]: layer i+1 is done reading it; ev_done[i]: layer i's
  // latest chapter is finished
  std::vector<cudaEvent_t> ev_pub[2], ev_read[2], ev_done;
  cudaEvent_t ev_start = nullptr;
  int device = 0;
};

namespace {

using ff::cuda_status;

int n_batches(const ff_pff_config& c) { return (c.n_pairs + c.batch_pairs - 1) / c.batch_pairs; }

float lr_at(float lr0, int epoch, int total, float cooldown_start) {
  if (!(cooldown_start < 1.f)) return lr0;
  const double e0 = (double)cooldown_start * total;
  if (epoch < e0) return lr0;
  return (float)((double)lr0 * (total - epoch) / (total - e0));
}

void release(ff_pff* p) {
  for (auto st : p->streams)
    if (st) {
      cudaStreamSynchronize(st);
      cudaStreamDestroy(st);
    }
  for (int s = 0; s < 2; ++s) {
    for (auto e : p->ev_pub[s])
      if (e) cudaEventDestroy(e);
    for (auto e : p->ev_read[s])
      if (e) cudaEventDestroy(e);
  }
  for (auto e : p->ev_done)
    if (e) cudaEventDestroy(e);
  if (p->ev_start) cudaEventDestroy(p->ev_start);
  ff::dev_free(p->pub_mem);
  for (auto* L : p->layers)
    if (L) L->last_stream = nullptr;  // its streams are gone
}

// Layer i's chapter c (global index) on stream st: C epochs of train steps,
// then (below the top layer) the published forward pass.
ff_status run_layer_chapter(ff_pff* p, int i, int c, int first, const float* x, const int* labels, float* loss,
                            cudaStream_t st) {
  const ff_pff_config& cf = p->cfg;
  ff_layer* L = p->layers[i];
  const int nl = (int)p->layers.size();
  const int slot = c & 1;
  const int nb = n_batches(cf);
  const int E = cf.epochs_per_chapter * cf.chapters;
  FF_TRY(cudaStreamWaitEvent(st, p->ev_done[i], 0), "layer order");
  if (i > 0) FF_TRY(cudaStreamWaitEvent(st, p->ev_pub[slot][i - 1], 0), "input ready");
  if (i + 1 < nl) FF_TRY(cudaStreamWaitEvent(st, p->ev_read[slot][i], 0), "output slot free");
  const int* lab = labels + (size_t)(c - first) * 2 * cf.n_pairs;
  const int ldin = i == 0 ? L->K : L->ldK;
  const size_t es = L->is_bf16 ? 2 : 4;
  auto input_rows = [&](int r0) -> const void* {
    if (i == 0) return x + (size_t)r0 * ldin;
    return static_cast<const char*>(p->pub[slot][i - 1]) + (size_t)r0 * ldin * es;
  };
  for (int m = 0; m < cf.epochs_per_chapter; ++m) {
    L->cfg.lr = lr_at(p->lr0[i], c * cf.epochs_per_chapter + m, E, cf.cooldown_start);
    for (int j = 0; j < nb; ++j) {
      const int r0 = 2 * j * cf.batch_pairs;
      const int b = (j + 1 < nb) ? cf.batch_pairs : cf.n_pairs - j * cf.batch_pairs;
      float* lp = loss ? loss + (((size_t)(c - first) * nl + i) * cf.epochs_per_chapter + m) * nb + j : nullptr;
      ff_status s = ff::train_step_impl(L, input_rows(r0), i == 0 ? lab + r0 : nullptr,
                                        i == 0 ? nullptr : p->pubs[slot][i - 1] + r0, b, nullptr, nullptr, nullptr,
                                        lp, st, nullptr, nullptr);
      if (s != FF_OK) return s;
    }
  }
  L->cfg.lr = p->lr0[i];
  if (i + 1 < nl) {
    const size_t eo = L->is_bf16 ? 2 : 4;
    for (int j = 0; j < nb; ++j) {
      const int r0 = 2 * j * cf.batch_pairs;
      const int rows = 2 * ((j + 1 < nb) ? cf.batch_pairs : cf.n_pairs - j * cf.batch_pairs);
      void* h = static_cast<char*>(p->pub[slot][i]) + (size_t)r0 * L->ldN * eo;
      ff_status s = ff_layer_forward(L, input_rows(r0), i == 0 ? lab + r0 : nullptr,
                                     i == 0 ? nullptr : p->pubs[slot][i - 1] + r0, rows, h, p->pubs[slot][i] + r0,
                                     nullptr, st);
      if (s != FF_OK) return s;
    }
    FF_TRY(cudaEventRecord(p->ev_pub[slot][i], st), "publish");
  }
  if (i > 0) FF_TRY(cudaEventRecord(p->ev_read[slot][i - 1], st), "input released");
  FF_TRY(cudaEventRecord(p->ev_done[i], st), "chapter done");
  return FF_OK;
}

}  // namespace

extern "C" {

ff_status ff_pff_create(ff_layer* const* layers, int n_layers, const ff_pff_config* cfg, ff_pff** out) {
  if (!out) return FF_ERR_INVALID_ARG;
  *out = nullptr;
  if (!layers || n_layers < 1 || !cfg) return FF_ERR_INVALID_ARG;
  if (cfg->n_pairs < 1 || cfg->batch_pairs < 1 || cfg->epochs_per_chapter < 1 || cfg->chapters < 1)
    return FF_ERR_INVALID_ARG;
  if (cfg->mode != FF_PFF_SINGLE_LAYER && cfg->mode != FF_PFF_ALL_LAYERS) return FF_ERR_INVALID_ARG;
  if (cfg->mode == FF_PFF_ALL_LAYERS && cfg->nodes < 1) return FF_ERR_INVALID_ARG;
  if (!std::isfinite(cfg->cooldown_start) || cfg->cooldown_start < 0.f) return FF_ERR_INVALID_ARG;
  for (int k = 0; k < n_layers; ++k) {
    if (!layers[k]) return FF_ERR_INVALID_ARG;
    if (layers[k]->is_bf16 != layers[0]->is_bf16) return FF_ERR_INVALID_ARG;
    if (k > 0 && layers[k]->K != layers[k - 1]->N) return FF_ERR_INVALID_ARG;
    for (int j = 0; j < k; ++j)
      if (layers[j] == layers[k]) return FF_ERR_INVALID_ARG;
  }
  if (layers[0]->K < 10) return FF_ERR_INVALID_ARG;
  ff_pff* p = new (std::nothrow) ff_pff();
  if (!p) return FF_ERR_OOM;
  p->cfg = *cfg;
  cudaGetDevice(&p->device);
  p->layers.assign(layers, layers + n_layers);
  for (auto* L : p->layers) p->lr0.push_back(L->cfg.lr);
  ff_status s = FF_OK;
  const int ns = cfg->mode == FF_PFF_SINGLE_LAYER ? n_layers : cfg->nodes;
  for (int k = 0; k < ns && s == FF_OK; ++k) {
    cudaStream_t st = nullptr;
    s = cuda_status(cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking), "pff stream");
    p->streams.push_back(st);
  }
  auto mkev = [&](std::vector<cudaEvent_t>& v, int n) {
    for (int k = 0; k < n && s == FF_OK; ++k) {
      cudaEvent_t e = nullptr;
      s = cuda_status(cudaEventCreateWithFlags(&e, cudaEventDisableTiming), "pff event");
      v.push_back(e);
    }
  };
  for (int sl = 0; sl < 2; ++sl) {
    mkev(p->ev_pub[sl], n_layers);
    mkev(p->ev_read[sl], n_layers);
  }
  mkev(p->ev_done, n_layers);
  if (s == FF_OK) s = cuda_status(cudaEventCreateWithFlags(&p->ev_start, cudaEventDisableTiming), "pff event");
  // published outputs: two chapter slots of [2P, ldN] activity + [2P] scale per layer below the top
  const size_t rows = 2 * (size_t)cfg->n_pairs;
  size_t bytes = 0;
  std::vector<size_t> offs;
  for (int k = 0; k + 1 < n_layers; ++k)
    for (int sl = 0; sl < 2; ++sl) {
      const size_t es = p->layers[k]->is_bf16 ? 2 : 4;
      offs.push_back(bytes);
      bytes += (rows * p->layers[k]->ldN * es + 255) & ~size_t(255);
      offs.push_back(bytes);
      bytes += (rows * 4 + 255) & ~size_t(255);
    }
  if (s == FF_OK && bytes) s = cuda_status(ff::dev_alloc(&p->pub_mem, bytes), "published outputs");
  for (int sl = 0; sl < 2; ++sl) {
    p->pub[sl].assign(n_layers, nullptr);
    p->pubs[sl].assign(n_layers, nullptr);
  }
  if (s == FF_OK) {
    size_t q = 0;
    char* base = static_cast<char*>(p->pub_mem);
    for (int k = 0; k + 1 < n_layers; ++k)
      for (int sl = 0; sl < 2; ++sl) {
        p->pub[sl][k] = base + offs[q++];
        p->pubs[sl][k] = reinterpret_cast<float*>(base + offs[q++]);
      }
  }
  // every layer's workspace sized for a whole batch now, never mid-run
  for (int k = 0; k < n_layers && s == FF_OK; ++k) s = ff::ensure_capacity(p->layers[k], 2 * cfg->batch_pairs);
  if (s != FF_OK) {
    release(p);
    delete p;
    return s;
  }
  *out = p;
  return FF_OK;
}

ff_status ff_pff_destroy(ff_pff* p) {
  if (!p) return FF_OK;
  release(p);
  delete p;
  return FF_OK;
}

ff_status ff_pff_run(ff_pff* p, const float* x, const int* labels, int first, int count, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_pff_run");
  if (!p || first < 0 || count < 0 || first + count > p->cfg.chapters) return FF_ERR_INVALID_ARG;
  if (count == 0) return FF_OK;
  if (!x || !labels) return FF_ERR_INVALID_ARG;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const int nl = (int)p->layers.size();
  // nothing starts before the caller's stream reaches this point
  FF_TRY(cudaEventRecord(p->ev_start, cs), "run start");
  for (auto st : p->streams) FF_TRY(cudaStreamWaitEvent(st, p->ev_start, 0), "run start");
  // wavefront: layer i's chapter c in step t = (c - first) + i
  for (int t = 0; t < count + nl - 1; ++t) {
    for (int i = 0; i < nl; ++i) {
      const int cc = t - i;
      if (cc < 0 || cc >= count) continue;
      const int c = first + cc;
      cudaStream_t st = p->cfg.mode == FF_PFF_SINGLE_LAYER ? p->streams[i] : p->streams[c % p->cfg.nodes];
      ff_status s = run_layer_chapter(p, i, c, first, x, labels, loss, st);
      if (s != FF_OK) return s;
    }
  }
  // the caller's stream waits for every layer's last chapter
  for (int i = 0; i < nl; ++i) FF_TRY(cudaStreamWaitEvent(cs, p->ev_done[i], 0), "run end");
  return FF_OK;
}

ff_status ff_pff_wait(ff_pff* p, unsigned timeout_ms) {
  if (!p) return FF_ERR_INVALID_ARG;
  std::vector<cudaEvent_t> evs;
  for (size_t k = 0; k < p->streams.size(); ++k) {
    cudaEvent_t e = nullptr;
    ff_status s = cuda_status(cudaEventCreateWithFlags(&e, cudaEventDisableTiming), "pff wait");
    if (s == FF_OK) s = cuda_status(cudaEventRecord(e, p->streams[k]), "pff wait");
    if (s != FF_OK) {
      if (e) cudaEventDestroy(e);
      for (auto x : evs) cudaEventDestroy(x);
      return s;
    }
    evs.push_back(e);
  }
  ff_status s = ff::wait_events(evs.data(), (int)evs.size(), timeout_ms);
  for (auto x : evs) cudaEventDestroy(x);
  return s;
}

}  // extern "C"
