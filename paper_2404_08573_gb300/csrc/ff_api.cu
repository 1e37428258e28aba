// The libff C ABI: FF layer lifecycle, the layer-local train step, the
// forward pass L_i(x), goodness prediction, and state access.  Host code only
// orchestrates; every step of the path runs in the kernels of ff_elem.cu,
// ff_gemm_tc.cu (bf16 mode) and ff_gemm_simt.cu (fp32 mode).
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <chrono>
#include <new>
#include <thread>

#include "ff_api_internal.h"
#include "ff_internal.cuh"
#include "ff_prof.h"

namespace ff {

static bool debug_enabled() {
  static const bool on = std::getenv("FF_DEBUG") != nullptr;
  return on;
}

ff_status cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return FF_OK;
  if (debug_enabled()) std::fprintf(stderr, "libff: %s: %s\n", what, cudaGetErrorString(e));
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return FF_ERR_OOM;
  }
  return FF_ERR_CUDA;
}


// Host-side fault injection: FF_FAULT_ALLOC_FAIL_AT=n makes the n-th device
// allocation (1-based, counted over the process) fail as out-of-memory.
cudaError_t dev_alloc(void** p, size_t bytes) {
  static long long fail_at = [] {
    const char* e = std::getenv("FF_FAULT_ALLOC_FAIL_AT");
    return e ? std::atoll(e) : 0ll;
  }();
  static long long count = 0;
  ++count;
  if (fail_at > 0 && count == fail_at) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  if (bytes == 0) bytes = 256;
  return cudaMalloc(p, bytes);
}

void dev_free(void* p) {
  if (p) cudaFree(p);
}

static size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

// goodness partials per row: the most either forward GEMM writes
static int gpart_tiles_max(int N) {
  const int a = tc_fwd_ntiles_max(N), b = simt_fwd_ntiles(N);
  return a > b ? a : b;
}

ff_status wait_events(const cudaEvent_t* ev, int n, unsigned timeout_ms) {
  const auto deadline = std::chrono::steady_clock::now() + std::chrono::milliseconds(timeout_ms);
  for (int k = 0; k < n;) {
    const cudaError_t e = cudaEventQuery(ev[k]);
    if (e == cudaSuccess) {
      ++k;
      continue;
    }
    if (e != cudaErrorNotReady) return cuda_status(e, "event query");
    if (std::chrono::steady_clock::now() >= deadline) return FF_ERR_TIMEOUT;
    std::this_thread::sleep_for(std::chrono::microseconds(50));
  }
  return FF_OK;
}

// Grows the per-row workspace to at least `rows` rows (one allocation).
ff_status ensure_capacity(ff_layer* L, int rows) {
  if (rows <= L->cap) return FF_OK;
  const int cap = ((rows + 127) / 128) * 128;
  const size_t es = L->is_bf16 ? 2 : 4;
  size_t off = 0;
  const size_t oX = off; off += align256((size_t)cap * L->ldK * es);
  const size_t oS = off; off += align256((size_t)cap * 4);
  const size_t oH = off; off += align256((size_t)cap * L->ldN * es);
  const size_t oZ = off; off += align256((size_t)cap * L->ldN * es);
  const size_t oP = off; off += align256((size_t)gpart_tiles_max(L->N) * cap * 4);
  const size_t oG = off; off += align256((size_t)cap * 4);
  const size_t oC = off; off += align256((size_t)cap * 4);
  const size_t oN = off; off += align256((size_t)cap * 4);
  const size_t oD = off; off += align256((size_t)local_grad_row_blocks(cap) * L->N * 4);
  const size_t oL = off; off += align256((size_t)(finalize_grid(cap) > local_grad_row_blocks(cap) ? finalize_grid(cap) : local_grad_row_blocks(cap)) * 4);
  const size_t oT = off; off += align256((size_t)local_grad_row_blocks(cap) * (2 + cdiv(L->ldN, 256)) * 4);
  if (L->cap > 0) {
    FF_TRY(cudaStreamSynchronize(L->last_stream), "sync before workspace growth");
    dev_free(L->X);
    L->X = nullptr;
    L->cap = 0;
  }
  void* base = nullptr;
  FF_TRY(dev_alloc(&base, off), "workspace allocation");
  char* b = static_cast<char*>(base);
  L->X = b + oX;
  L->s_in = reinterpret_cast<float*>(b + oS);
  L->H = b + oH;
  L->dZ = b + oZ;
  L->gpart = reinterpret_cast<float*>(b + oP);
  L->g = reinterpret_cast<float*>(b + oG);
  L->c = reinterpret_cast<float*>(b + oC);
  L->s_next = reinterpret_cast<float*>(b + oN);
  L->dbpart = reinterpret_cast<float*>(b + oD);
  L->loss_part = reinterpret_cast<float*>(b + oL);
  L->stat_part = reinterpret_cast<float*>(b + oT);
  L->cap = cap;
  return FF_OK;
}

static void free_layer(ff_layer* L) {
  if (!L) return;
  dev_free(L->kpart);
  dev_free(L->kcnt);
  dev_free(L->W);
  dev_free(L->mW);  // also holds v_W
  dev_free(L->dW);
  dev_free(L->b);
  dev_free(L->Wb);
  dev_free(L->ds);
  dev_free(L->X);
  dev_free(L->pws);
  delete L;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Forward pass of one layer on M rows: operand preparation, the GEMM with the
// fused scale/bias/ReLU/goodness epilogue.  Leaves per-tile goodness partials
// in L->gpart and reports the row scale, activity buffer, operand buffer and
// number of partial tiles it used.
struct FwdResult {
  const float* s;
  void* H;
  const void* X;
  int ntiles;
  bool local_grad_done;  // the forward's epilogue also formed the local step (tc_gemm_fwd_lg)
};

// Split-K scratch of an fp32 layer's forward and weight-gradient GEMMs on M
// rows (grown on demand; new counters start at zero).
static ff_status ensure_split(ff_layer* L, int M) {
  const size_t fwd = simt_split_floats(M, L->N, L->K), wg = simt_split_floats(L->N, L->K, M);
  const size_t need = fwd > wg ? fwd : wg;
  if (need == 0) return FF_OK;
  const int t1 = simt_split_tiles(M, L->N), t2 = simt_split_tiles(L->N, L->K);
  const int tiles = t1 > t2 ? t1 : t2;
  if (need <= L->kpart_cap && tiles <= L->kcnt_cap) return FF_OK;
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync before split scratch growth");
  dev_free(L->kpart);
  dev_free(L->kcnt);
  L->kpart = nullptr;
  L->kcnt = nullptr;
  L->kpart_cap = 0;
  L->kcnt_cap = 0;
  FF_TRY(dev_alloc(reinterpret_cast<void**>(&L->kpart), need * sizeof(float)), "split scratch");
  FF_TRY(dev_alloc(reinterpret_cast<void**>(&L->kcnt), (size_t)tiles * sizeof(int)), "split counters");
  FF_TRY(cudaMemset(L->kcnt, 0, (size_t)tiles * sizeof(int)), "zero split counters");
  L->kpart_cap = need;
  L->kcnt_cap = tiles;
  return FF_OK;
}

// x_rows: rows of the raw input x when labels are given (0: M; M / 2: one
// image per pair, read for the positive and the negative row).
// lg (train steps): the local step's arguments; for a bf16 layer whose shape
// allows it, the forward GEMM forms that step in its epilogue as well
// (r->local_grad_done), with lg->s set to the row scale used here.
static ff_status forward_core(ff_layer* L, const void* x, const int* labels, const float* row_scale, int M,
                              void* h_out, cudaStream_t st, cudaEvent_t ev_input_read, FwdResult* r,
                              int x_rows = 0, GradPrepArgs* lg = nullptr) {
  const int K = L->K, N = L->N;
  if (!L->is_bf16) {
    const ff_status ss = ensure_split(L, M);
    if (ss != FF_OK) return ss;
  }
  const double es = L->is_bf16 ? 2.0 : 4.0;
  const float* s;
  const void* X;
  if (labels) {
    FF_LAUNCH(K_OVERLAY, (double)M * (K * 4.0 + L->ldK * es + 8), st,
              launch_overlay(static_cast<const float*>(x), labels, M, K, L->X, L->ldK, L->is_bf16, L->s_in, 0, st,
                             x_rows),
              "overlay");
    if (ev_input_read) FF_TRY(cudaEventRecord(ev_input_read, st), "event record");
    X = L->X;
    s = L->s_in;
  } else {
    X = x;
    if (row_scale) {
      s = row_scale;
    } else {
      FF_LAUNCH(K_ROW_SCALE, (double)M * (K * es + 4), st, launch_row_scale(x, L->ldK, L->is_bf16, M, K, L->s_in, st),
                "row scale");
      s = L->s_in;
    }
  }
  void* H = h_out ? h_out : L->H;
  EpiArgs ep{s, L->cfg.has_bias ? L->b : nullptr, H, L->ldN, L->gpart};
  int ntiles;
  r->local_grad_done = false;
  if (L->is_bf16 && lg && L->fuse_local_grad && tc_fwd_lg_supported(M, N)) {
    ntiles = tc_fwd_ntiles(M, N, false);
    lg->s = s;
    ep.gpart = nullptr;
    FF_LAUNCH(K_FWD_TC, 2.0 * M * N * K, st,
              tc_gemm_fwd_lg(static_cast<const bf16*>(X), L->ldK, L->Wb, L->ldK, M, N, K, ep, *lg,
                             static_cast<bf16*>(L->dZ), &L->ds->err, st),
              "forward GEMM with the local gradient (tcgen05)");
    r->local_grad_done = true;
  } else if (L->is_bf16) {
    ntiles = tc_fwd_ntiles(M, N, false);
    FF_LAUNCH(K_FWD_TC, 2.0 * M * N * K, st,
              tc_gemm_fwd(static_cast<const bf16*>(X), L->ldK, L->Wb, L->ldK, M, N, K, ep, &L->ds->err, st),
              "forward GEMM (tcgen05)");
  } else {
    ntiles = simt_fwd_ntiles(N);
    ep.kpart = L->kpart;
    ep.kpart_cap = L->kpart_cap;
    ep.kcnt = L->kcnt;
    ep.kcnt_cap = L->kcnt_cap;
    FF_LAUNCH(K_FWD_SIMT, 2.0 * M * N * K, st,
              simt_gemm_fwd(static_cast<const float*>(X), L->ldK, L->W, K, M, N, K, ep, st), "forward GEMM (fp32)");
  }
  r->s = s;
  r->H = H;
  r->X = X;
  r->ntiles = ntiles;
  return FF_OK;
}

static ff_status check_call(ff_layer* L, const void* x, const int* labels, int rows) {
  if (!L || !x || rows < 0) return FF_ERR_INVALID_ARG;
  if (labels && L->K < 10) return FF_ERR_INVALID_ARG;
  if (!labels && !aligned16(x)) return FF_ERR_INVALID_ARG;
  if (labels && (reinterpret_cast<uintptr_t>(x) & 3u)) return FF_ERR_INVALID_ARG;
  return FF_OK;
}

ff_status train_step_impl(ff_layer* L, const void* x, const int* labels, const float* row_scale, int B, void* h_out,
                          float* next_scale, float* goodness, float* loss, cudaStream_t st,
                          cudaEvent_t ev_input_read, cudaEvent_t ev_forward_done, bool images_once) {
  ff_status cs = check_call(L, x, labels, B);
  if (cs != FF_OK) return cs;
  if (h_out && !aligned16(h_out)) return FF_ERR_INVALID_ARG;
  if (B == 0) return FF_OK;
  const int M = 2 * B;
  if (M < B) return FF_ERR_INVALID_ARG;
  ff_status cap_st = ensure_capacity(L, M);
  if (cap_st != FF_OK) return cap_st;
  L->last_stream = st;
  const double es = L->is_bf16 ? 2.0 : 4.0;
  GradPrepArgs ga{};
  ga.gpart = L->gpart;
  ga.M = M;
  ga.N = L->N;
  ga.ld = L->ldN;
  ga.B = B;
  ga.theta = L->cfg.theta;
  ga.g_out = goodness;
  ga.s_next = next_scale;
  ga.dbpart = L->dbpart;
  ga.loss_part = L->loss_part;
  ga.stat_part = L->stat_part;
  ga.ncb = cdiv(L->ldN, 256);
  ga.ds = L->ds;
  ga.beta1 = L->cfg.beta1;
  ga.beta2 = L->cfg.beta2;
  ga.err = &L->ds->err;
  FwdResult fr;
  ff_status fs = forward_core(L, x, labels, row_scale, M, h_out, st, ev_input_read, &fr,
                              images_once && labels ? B : 0, &ga);
  if (fs != FF_OK) return fs;
  if (!fr.local_grad_done) {
    ga.ntiles = fr.ntiles;
    ga.s = fr.s;
    FF_LAUNCH(K_GRAD_PREP,
              (double)M * (fr.ntiles * 4.0 + 12) + (double)M * L->ldN * es * 2 + (double)local_grad_row_blocks(M) * L->N * 4,
              st, launch_grad_prep(ga, L->is_bf16, fr.H, L->dZ, st), "goodness/loss/local gradient");
  }
  if (ev_forward_done) FF_TRY(cudaEventRecord(ev_forward_done, st), "event record");

  if (L->is_bf16) {
    FF_LAUNCH(K_WGRAD_TC, 2.0 * M * L->N * L->K, st,
              tc_gemm_wgrad(static_cast<const bf16*>(L->dZ), L->ldN, static_cast<const bf16*>(fr.X), L->ldK, M,
                            L->N, L->K, L->dW, L->K, &L->ds->err, st),
              "weight-gradient GEMM (tcgen05)");
  } else {
    EpiArgs split{};
    split.kpart = L->kpart;
    split.kpart_cap = L->kpart_cap;
    split.kcnt = L->kcnt;
    split.kcnt_cap = L->kcnt_cap;
    FF_LAUNCH(K_WGRAD_SIMT, 2.0 * M * L->N * L->K, st,
              simt_gemm_wgrad(static_cast<const float*>(L->dZ), L->ldN, static_cast<const float*>(fr.X), L->ldK, M,
                              L->N, L->K, L->dW, L->K, st, &split),
              "weight-gradient GEMM (fp32)");
  }
  AdamArgs aa{};
  aa.W = L->W;
  aa.mW = L->mW;
  aa.vW = L->vW;
  aa.dW = L->dW;
  aa.N = L->N;
  aa.K = L->K;
  aa.Wb = L->is_bf16 ? L->Wb : nullptr;
  aa.ldb = L->ldK;
  aa.b = L->b;
  aa.mb = L->mb;
  aa.vb = L->vb;
  aa.dbpart = L->dbpart;
  aa.nrb = local_grad_row_blocks(M);
  aa.db_out = L->db;
  aa.has_bias = L->cfg.has_bias;
  aa.lr = L->cfg.lr;
  aa.beta1 = L->cfg.beta1;
  aa.beta2 = L->cfg.beta2;
  aa.eps = L->cfg.eps;
  aa.ds = L->ds;
  aa.loss_part = L->loss_part;
  aa.stat_part = L->stat_part;
  aa.ncb = cdiv(L->ldN, 256);
  aa.stats_out = L->ds->stats;
  aa.loss_out = loss ? loss : &L->ds->loss;
  aa.B = B;
  // Data nobody reads after this step, so its dirty lines need not reach HBM:
  // dW (unless kept for ff_layer_get_grad) and the local-gradient operand.
  // (Dropping the activities' lines as well measured no further gain.)
  aa.discard_dW = !L->cfg.keep_grad && ((uintptr_t)L->dW & 127u) == 0;
  if (!L->cfg.keep_grad) add_dead(aa, L->dZ, (size_t)M * L->ldN * (size_t)es);
  FF_LAUNCH(K_ADAM, (double)L->N * L->K * (28.0 + (L->is_bf16 ? 2.0 : 0.0)) + (double)L->N * (aa.nrb * 4.0 + 28), st,
            launch_adam(aa, st),
            "Adam");
  return FF_OK;
}

}  // namespace ff

using namespace ff;

extern "C" {

const char* ff_status_string(ff_status s) {
  switch (s) {
    case FF_OK: return "FF_OK";
    case FF_ERR_INVALID_ARG: return "FF_ERR_INVALID_ARG";
    case FF_ERR_CUDA: return "FF_ERR_CUDA";
    case FF_ERR_OOM: return "FF_ERR_OOM";
    case FF_ERR_TIMEOUT: return "FF_ERR_TIMEOUT";
    case FF_ERR_NONFINITE: return "FF_ERR_NONFINITE";
    case FF_ERR_UNSUPPORTED: return "FF_ERR_UNSUPPORTED";
    case FF_ERR_DEVICE_CHECK: return "FF_ERR_DEVICE_CHECK";
  }
  return "FF_ERR_UNKNOWN";
}

int ff_row_stride(int features) { return features <= 0 ? 0 : ff::row_stride(features); }

ff_status ff_layer_create(const ff_layer_config* cfg, void* stream, ff_layer** out) {
  if (!out) return FF_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || cfg->in_features < 1 || cfg->out_features < 1 || cfg->max_rows < 0) return FF_ERR_INVALID_ARG;
  if (cfg->prec != FF_FP32 && cfg->prec != FF_BF16) return FF_ERR_INVALID_ARG;
  if (!std::isfinite(cfg->theta) || !std::isfinite(cfg->lr) || !(cfg->beta1 >= 0.f && cfg->beta1 < 1.f) ||
      !(cfg->beta2 >= 0.f && cfg->beta2 < 1.f) || !(cfg->eps >= 0.f))
    return FF_ERR_INVALID_ARG;
  if ((long long)cfg->in_features * cfg->out_features > (1ll << 40)) return FF_ERR_INVALID_ARG;
  int dev = 0;
  FF_TRY(cudaGetDevice(&dev), "cudaGetDevice");
  if (cfg->prec == FF_BF16 && !tc_supported()) return FF_ERR_UNSUPPORTED;
  ff_layer* L = new (std::nothrow) ff_layer();  // value-initialised: null pointers, zero sizes, defaults
  if (!L) return FF_ERR_OOM;
  L->cfg = *cfg;
  L->K = cfg->in_features;
  L->N = cfg->out_features;
  L->ldK = row_stride(L->K);
  L->ldN = row_stride(L->N);
  L->device = dev;
  L->is_bf16 = cfg->prec == FF_BF16;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  L->last_stream = st;
  const size_t nk = (size_t)L->N * L->K;
  ff_status s = FF_OK;
#define FF_ALLOC(ptr, bytes)                                                      \
  do {                                                                            \
    s = cuda_status(dev_alloc(reinterpret_cast<void**>(&(ptr)), (bytes)), #ptr); \
    if (s != FF_OK) {                                                             \
      free_layer(L);                                                              \
      return s;                                                                   \
    }                                                                             \
  } while (0)
  FF_ALLOC(L->W, nk * 4);
  FF_ALLOC(L->mW, nk * 4 * 2);  // m_W then v_W, one range
  L->vW = L->mW + nk;
  FF_ALLOC(L->dW, nk * 4);
  FF_ALLOC(L->b, (size_t)L->N * 4 * 4);  // b, mb, vb, db
  if (L->is_bf16) FF_ALLOC(L->Wb, (size_t)L->N * L->ldK * 2);
  FF_ALLOC(L->ds, sizeof(ff_dev_state));
#undef FF_ALLOC
  L->mb = L->b + L->N;
  L->vb = L->b + 2 * L->N;
  L->db = L->b + 3 * L->N;
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = cudaMemsetAsync(L->mW, 0, nk * 4, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(L->vW, 0, nk * 4, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(L->dW, 0, nk * 4, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(L->b, 0, (size_t)L->N * 4 * 4, st);
  if (e == cudaSuccess) {
    static const ff_dev_state fresh = {0, 1.0, 1.0, 0.f, 0.f, 0, 0.f};
    e = cudaMemcpyAsync(L->ds, &fresh, sizeof(ff_dev_state), cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // `fresh` is pageable host memory
  }
  if (e == cudaSuccess) {
    ProfScope p(K_INIT, (double)nk * 4, st);
    e = p.injected_failure() ? cudaErrorLaunchOutOfResources
                             : launch_init_weights(L->W, L->N, L->K, cfg->init_seed, st);
  }
  if (e == cudaSuccess && L->is_bf16) {
    ProfScope p(K_TO_BF16, (double)nk * 4 + (double)L->N * L->ldK * 2, st);
    e = p.injected_failure() ? cudaErrorLaunchOutOfResources
                             : launch_to_bf16(L->W, L->N, L->K, L->Wb, L->ldK, st);
  }
  s = cuda_status(e, "layer initialisation");
  if (s == FF_OK) s = ensure_capacity(L, cfg->max_rows > 0 ? cfg->max_rows : 256);
  if (s != FF_OK) {
    cudaStreamSynchronize(st);
    free_layer(L);
    return s;
  }
  *out = L;
  return FF_OK;
}

ff_status ff_layer_destroy(ff_layer* L) {
  if (!L) return FF_OK;
  cudaError_t e = cudaStreamSynchronize(L->last_stream);
  free_layer(L);
  return cuda_status(e, "destroy sync");
}

ff_status ff_overlay_label(const float* x, const int* labels, int rows, int features, void* out, float* row_scale,
                           ff_precision prec, void* stream) {
  ff::NvtxRange nvtx_("ff_overlay_label");
  if (rows < 0 || features < 10 || (prec != FF_FP32 && prec != FF_BF16)) return FF_ERR_INVALID_ARG;
  if (rows == 0) return FF_OK;
  if (!x || !labels || !out) return FF_ERR_INVALID_ARG;
  FF_LAUNCH(K_OVERLAY, (double)rows * (features * 4.0 + row_stride(features) * (prec == FF_BF16 ? 2.0 : 4.0) + 8),
            static_cast<cudaStream_t>(stream),
            launch_overlay(x, labels, rows, features, out, row_stride(features), prec == FF_BF16, row_scale, 0,
                           static_cast<cudaStream_t>(stream)),
            "overlay");
  return FF_OK;
}

ff_status ff_layer_forward(ff_layer* L, const void* x, const int* labels, const float* row_scale, int rows,
                           void* h_out, float* next_scale, float* goodness, void* stream) {
  ff::NvtxRange nvtx_("ff_layer_forward");
  ff_status cs = check_call(L, x, labels, rows);
  if (cs != FF_OK) return cs;
  if (!h_out && !next_scale && !goodness) return FF_ERR_INVALID_ARG;
  if (h_out && !aligned16(h_out)) return FF_ERR_INVALID_ARG;
  if (rows == 0) return FF_OK;
  ff_status es = ensure_capacity(L, rows);
  if (es != FF_OK) return es;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  L->last_stream = st;
  FwdResult fr;
  ff_status fs = forward_core(L, x, labels, row_scale, rows, h_out, st, nullptr, &fr);
  if (fs != FF_OK) return fs;
  FinalizeArgs fa{};
  fa.gpart = L->gpart;
  fa.ntiles = fr.ntiles;
  fa.M = rows;
  fa.g_out = goodness;
  fa.s_next = next_scale;
  fa.err = &L->ds->err;
  FF_LAUNCH(K_FINALIZE, (double)rows * (fr.ntiles * 4.0 + 8), st, launch_finalize(fa, st), "goodness");
  return FF_OK;
}

ff_status ff_layer_train_step(ff_layer* L, const void* x, const int* labels, const float* row_scale, int B,
                              void* h_out, float* next_scale, float* goodness, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_layer_train_step");
  return train_step_impl(L, x, labels, row_scale, B, h_out, next_scale, goodness, loss,
                         static_cast<cudaStream_t>(stream), nullptr, nullptr);
}

// Goodness prediction over the 10 label overlays (§3 "Prediction"); with
// `labels`, the argmax leaves each sample's own label out (AdaptiveNEG, §5).
static ff_status predict_impl(ff_layer* const* layers, int n_layers, const float* x, const int* labels, int n,
                              int* pred, float* goodness, cudaStream_t st) {
  if (!layers || n_layers < 1 || n < 0) return FF_ERR_INVALID_ARG;
  for (int k = 0; k < n_layers; ++k) {
    if (!layers[k]) return FF_ERR_INVALID_ARG;
    if (layers[k]->is_bf16 != layers[0]->is_bf16) return FF_ERR_INVALID_ARG;
    if (k > 0 && layers[k]->K != layers[k - 1]->N) return FF_ERR_INVALID_ARG;
  }
  if (n == 0) return FF_OK;
  if (!x || !pred) return FF_ERR_INVALID_ARG;
  ff_layer* L0 = layers[0];
  if (L0->K < 10) return FF_ERR_INVALID_ARG;
  const bool b16 = L0->is_bf16;
  const size_t es = b16 ? 2 : 4;
  // fp32 layers: the GEMMs on the tensor cores (three TF32 products) where
  // every layer's rows allow TMA, else on the CUDA cores
  bool f32tc = !b16;
  for (int k = 0; k < n_layers && f32tc; ++k) f32tc = tc_f32_supported(layers[k]->K, layers[k]->ldK, layers[k]->K);
  int ldmax = 0, ntmax = 0;
  for (int k = 0; k < n_layers; ++k) {
    if (layers[k]->ldN > ldmax) ldmax = layers[k]->ldN;
    const int nt = b16 || f32tc ? tc_fwd_ntiles_max(layers[k]->N) : simt_fwd_ntiles(layers[k]->N);
    if (nt > ntmax) ntmax = nt;
  }
  // Samples per chunk: about 40 MB of activations per buffer, so that one
  // chunk's two activation buffers stay resident in L2 between layers.
  long long per = (40ll << 20) / ((long long)10 * ldmax * es);
  int C = (int)(per < 64 ? 64 : per > 8192 ? 8192 : per);
  if ((b16 || f32tc) && n > C) {
    // Each forward GEMM CTA holds a whole SM, so a chunk whose GEMMs end in a
    // nearly empty last wave wastes most of that wave: among chunk sizes
    // down to half the L2 budget, take the one whose widest hidden GEMM fills
    // its waves best (the largest on ties).  (fp32 forward GEMMs never narrow
    // their tiles.)
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) ==
                                                   cudaSuccess && sms > 0 && n_layers > 1) {
      int Nw = 0;
      for (int k = 1; k < n_layers; ++k)
        if (layers[k]->N > Nw) Nw = layers[k]->N;
      double best = -1.0;
      int bestC = C;
      for (int c = C; c >= C / 2 && c >= 64; --c) {
        const int ctas = tc_gemm_fwd_ctas(10 * c, Nw, b16);
        const double eff = (double)ctas / ((double)cdiv(ctas, sms) * sms);
        if (eff > best + 1e-9) {
          best = eff;
          bestC = c;
        }
      }
      C = bestC;
    }
  }
  if (C > n) C = n;
  const int R = 10 * C;
  const int N1 = L0->N;
  size_t off = 0;
  const size_t oX = off; off += align256((size_t)C * L0->ldK * es);
  const size_t oS1 = off; off += align256((size_t)C * 4);
  const size_t oBase = off; off += align256((size_t)C * L0->ldN * 4);
  const size_t oCols = off; off += align256((size_t)10 * L0->ldN * 4);
  const size_t oH0 = off; off += align256((size_t)R * ldmax * es);
  const size_t oH1 = off; off += align256((size_t)R * ldmax * es);
  const size_t oSa = off; off += align256((size_t)R * 4);
  const size_t oSb = off; off += align256((size_t)R * 4);
  const size_t oP = off; off += align256((size_t)ntmax * R * 4);
  const size_t oP2 = off; off += align256(b16 ? (size_t)ntmax * R * 4 : 0);
  const size_t oG = off; off += align256(goodness ? 0 : (size_t)n * 10 * 4);
  if (off > L0->pws_bytes) {
    FF_TRY(cudaStreamSynchronize(L0->last_stream), "sync before predict scratch growth");
    dev_free(L0->pws);
    L0->pws = nullptr;
    L0->pws_bytes = 0;
    FF_TRY(dev_alloc(&L0->pws, off), "predict scratch");
    L0->pws_bytes = off;
  }
  L0->last_stream = st;
  char* w = static_cast<char*>(L0->pws);
  void* X0 = w + oX;
  float* s1 = reinterpret_cast<float*>(w + oS1);
  float* base = reinterpret_cast<float*>(w + oBase);
  float* cols = reinterpret_cast<float*>(w + oCols);
  void* Hb[2] = {w + oH0, w + oH1};
  float* Sb[2] = {reinterpret_cast<float*>(w + oSa), reinterpret_cast<float*>(w + oSb)};
  // goodness partials of the forward GEMMs, alternating between layers on the
  // tensor-core path (a GEMM reads the previous layer's while writing its own)
  float* gpb[2] = {reinterpret_cast<float*>(w + oP), reinterpret_cast<float*>(w + (b16 ? oP2 : oP))};
  float* G = goodness ? goodness : reinterpret_cast<float*>(w + oG);
  int* err = &L0->ds->err;

  FF_TRY(cudaMemsetAsync(G, 0, (size_t)n * 10 * 4, st), "zero goodness");
  FF_LAUNCH(K_LABEL_COLS, (double)N1 * 10 * (es + 4), st,
            launch_label_columns(b16 ? (const void*)L0->Wb : (const void*)L0->W, b16 ? L0->ldK : L0->K, b16, N1,
                                 cols, L0->ldN, st),
            "label columns");
  for (int c0 = 0; c0 < n; c0 += C) {
    const int cn = (n - c0) < C ? (n - c0) : C;
    const int rows = 10 * cn;
    FF_LAUNCH(K_OVERLAY, (double)cn * (L0->K * 4.0 + L0->ldK * es + 4), st,
              launch_overlay(x + (size_t)c0 * L0->K, nullptr, cn, L0->K, X0, L0->ldK, b16, s1, 1, st),
              "zero label area");
    if (b16) {
      FF_LAUNCH(K_STORE_TC, 2.0 * cn * N1 * L0->K, st,
                tc_gemm_store(static_cast<const bf16*>(X0), L0->ldK, L0->Wb, L0->ldK, cn, N1, L0->K, base, L0->ldN,
                              err, st),
                "layer-1 base GEMM (tcgen05)");
    } else if (f32tc) {
      FF_LAUNCH(K_STORE_TC, 2.0 * cn * N1 * L0->K, st,
                tc_gemm_store_f32(static_cast<const float*>(X0), L0->ldK, L0->W, L0->K, cn, N1, L0->K, base,
                                  L0->ldN, err, st),
                "layer-1 base GEMM (fp32, tcgen05 TF32 x 3)");
    } else {
      FF_LAUNCH(K_STORE_SIMT, 2.0 * cn * N1 * L0->K, st,
                simt_gemm_store(static_cast<const float*>(X0), L0->ldK, L0->W, L0->K, cn, N1, L0->K, base, L0->ldN,
                                st),
                "layer-1 base GEMM (fp32)");
    }
    float* Gc = G + (size_t)c0 * 10;
    FF_LAUNCH(K_EXPAND, (double)cn * (L0->ldN * 4.0 + 10.0 * L0->ldN * es + 40), st,
              launch_expand(base, L0->ldN, cols, s1, L0->cfg.has_bias ? L0->b : nullptr, cn, N1, Hb[0], L0->ldN, b16,
                            Sb[0], n_layers == 1 ? Gc : nullptr, err, st),
              "layer-1 expansion");
    int cur = 0;
    int nt_prev = 0;
    for (int k = 1; k < n_layers; ++k) {
      ff_layer* Lk = layers[k];
      float* gpart = gpb[k & 1];
      EpiArgs ep{Sb[cur], Lk->cfg.has_bias ? Lk->b : nullptr, Hb[cur ^ 1], Lk->ldN, gpart};
      ep.narrow = true;
      int nt;
      if (b16) {
        if (k >= 2) {
          // the row scale and layer k-1's share of G come from layer k-1's
          // goodness partials inside this GEMM (no separate finalize)
          ep.row_scale = nullptr;
          ep.gpart_in = gpb[(k - 1) & 1];
          ep.ntiles_in = nt_prev;
          ep.G_acc = Gc;
        }
        nt = tc_fwd_ntiles(rows, Lk->N, true);
        FF_LAUNCH(K_FWD_TC, 2.0 * rows * Lk->N * Lk->K, st,
                  tc_gemm_fwd(static_cast<const bf16*>(Hb[cur]), Lk->ldK, Lk->Wb, Lk->ldK, rows, Lk->N, Lk->K, ep,
                              err, st),
                  "predict forward GEMM (tcgen05)");
      } else if (f32tc) {
        ep.narrow = false;
        nt = tc_fwd_ntiles(rows, Lk->N, false);
        FF_LAUNCH(K_FWD_TC, 2.0 * rows * Lk->N * Lk->K, st,
                  tc_gemm_fwd_f32(static_cast<const float*>(Hb[cur]), Lk->ldK, Lk->W, Lk->K, rows, Lk->N, Lk->K, ep,
                                  err, st),
                  "predict forward GEMM (fp32, tcgen05 TF32 x 3)");
      } else {
        nt = simt_fwd_ntiles(Lk->N);
        FF_LAUNCH(K_FWD_SIMT, 2.0 * rows * Lk->N * Lk->K, st,
                  simt_gemm_fwd(static_cast<const float*>(Hb[cur]), Lk->ldK, Lk->W, Lk->K, rows, Lk->N, Lk->K, ep, st),
                  "predict forward GEMM (fp32)");
      }
      nt_prev = nt;
      if (!b16 || k + 1 == n_layers) {
        FinalizeArgs fa{};
        fa.gpart = gpart;
        fa.ntiles = nt;
        fa.M = rows;
        fa.s_next = (k + 1 < n_layers) ? Sb[cur ^ 1] : nullptr;
        fa.G_acc = Gc;
        fa.err = err;
        FF_LAUNCH(K_FINALIZE, (double)rows * (nt * 4.0 + 12), st, launch_finalize(fa, st), "predict goodness");
      }
      cur ^= 1;
    }
  }
  FF_LAUNCH(K_ARGMAX, (double)n * (labels ? 48 : 44), st, launch_argmax(G, n, labels, pred, st), "argmax");
  return FF_OK;
}

ff_status ff_predict(ff_layer* const* layers, int n_layers, const float* x, int n, int* pred, float* goodness,
                     void* stream) {
  ff::NvtxRange nvtx_("ff_predict");
  return predict_impl(layers, n_layers, x, nullptr, n, pred, goodness, static_cast<cudaStream_t>(stream));
}

ff_status ff_adaptive_negatives(ff_layer* const* layers, int n_layers, const float* x, const int* labels, int n,
                                int* neg, float* goodness, void* stream) {
  ff::NvtxRange nvtx_("ff_adaptive_negatives");
  if (n > 0 && !labels) return FF_ERR_INVALID_ARG;
  return predict_impl(layers, n_layers, x, labels, n, neg, goodness, static_cast<cudaStream_t>(stream));
}

static cudaMemcpyKind kind_default() { return cudaMemcpyDefault; }

ff_status ff_layer_get_state(const ff_layer* Lc, float* W, float* b, float* m_W, float* v_W, float* m_b, float* v_b,
                             long long* step) {
  if (!Lc) return FF_ERR_INVALID_ARG;
  ff_layer* L = const_cast<ff_layer*>(Lc);
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  const size_t nk = (size_t)L->N * L->K * 4, n4 = (size_t)L->N * 4;
  if (W) FF_TRY(cudaMemcpy(W, L->W, nk, kind_default()), "copy W");
  if (m_W) FF_TRY(cudaMemcpy(m_W, L->mW, nk, kind_default()), "copy m_W");
  if (v_W) FF_TRY(cudaMemcpy(v_W, L->vW, nk, kind_default()), "copy v_W");
  if (b) FF_TRY(cudaMemcpy(b, L->b, n4, kind_default()), "copy b");
  if (m_b) FF_TRY(cudaMemcpy(m_b, L->mb, n4, kind_default()), "copy m_b");
  if (v_b) FF_TRY(cudaMemcpy(v_b, L->vb, n4, kind_default()), "copy v_b");
  if (step) FF_TRY(cudaMemcpy(step, &L->ds->t, sizeof(long long), cudaMemcpyDeviceToHost), "copy step");
  return FF_OK;
}

ff_status ff_layer_set_state(ff_layer* L, const float* W, const float* b, const float* m_W, const float* v_W,
                             const float* m_b, const float* v_b, long long step) {
  if (!L || step < 0) return FF_ERR_INVALID_ARG;
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  const size_t nk = (size_t)L->N * L->K * 4, n4 = (size_t)L->N * 4;
  if (W) FF_TRY(cudaMemcpy(L->W, W, nk, kind_default()), "copy W");
  if (m_W) FF_TRY(cudaMemcpy(L->mW, m_W, nk, kind_default()), "copy m_W");
  if (v_W) FF_TRY(cudaMemcpy(L->vW, v_W, nk, kind_default()), "copy v_W");
  if (b) FF_TRY(cudaMemcpy(L->b, b, n4, kind_default()), "copy b");
  if (m_b) FF_TRY(cudaMemcpy(L->mb, m_b, n4, kind_default()), "copy m_b");
  if (v_b) FF_TRY(cudaMemcpy(L->vb, v_b, n4, kind_default()), "copy v_b");
  FF_TRY(cudaMemcpy(&L->ds->t, &step, sizeof(long long), cudaMemcpyHostToDevice), "copy step");
  const double pw[2] = {std::pow((double)L->cfg.beta1, (double)step), std::pow((double)L->cfg.beta2, (double)step)};
  FF_TRY(cudaMemcpy(&L->ds->pow1, pw, sizeof(pw), cudaMemcpyHostToDevice), "copy beta powers");
  if (L->is_bf16) {
    FF_LAUNCH(K_TO_BF16, (double)L->N * L->K * 4 + (double)L->N * L->ldK * 2, L->last_stream,
              launch_to_bf16(L->W, L->N, L->K, L->Wb, L->ldK, L->last_stream), "refresh bf16 W");
    FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  }
  return FF_OK;
}

ff_status ff_layer_get_grad(const ff_layer* Lc, float* dW, float* db) {
  if (!Lc) return FF_ERR_INVALID_ARG;
  if (!Lc->cfg.keep_grad) return FF_ERR_UNSUPPORTED;
  ff_layer* L = const_cast<ff_layer*>(Lc);
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  if (dW) FF_TRY(cudaMemcpy(dW, L->dW, (size_t)L->N * L->K * 4, kind_default()), "copy dW");
  if (db) FF_TRY(cudaMemcpy(db, L->db, (size_t)L->N * 4, kind_default()), "copy db");
  return FF_OK;
}

ff_status ff_layer_get_grad_operand(const ff_layer* Lc, void* out, int rows) {
  if (!Lc || !out || rows < 0) return FF_ERR_INVALID_ARG;
  if (!Lc->cfg.keep_grad) return FF_ERR_UNSUPPORTED;
  if (rows > Lc->cap) return FF_ERR_INVALID_ARG;
  ff_layer* L = const_cast<ff_layer*>(Lc);
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  if (rows) FF_TRY(cudaMemcpy(out, L->dZ, (size_t)rows * L->ldN * (L->is_bf16 ? 2 : 4), kind_default()), "copy G");
  return FF_OK;
}

ff_status ff_layer_selftest_wait(ff_layer* L, unsigned int timeout_us, void* stream) {
  if (!L || timeout_us == 0 || timeout_us > 10000000u) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  L->last_stream = st;
  FF_TRY(launch_wait_selftest(&L->ds->err, 1000ull * timeout_us, st), "bounded-wait self-test");
  return FF_OK;
}

ff_status ff_layer_get_stats(const ff_layer* Lc, float* stats) {
  if (!Lc || !stats) return FF_ERR_INVALID_ARG;
  ff_layer* L = const_cast<ff_layer*>(Lc);
  FF_TRY(cudaStreamSynchronize(L->last_stream), "sync");
  FF_TRY(cudaMemcpy(stats, L->ds->stats, 3 * sizeof(float), cudaMemcpyDefault), "read statistics");
  return FF_OK;
}

ff_status ff_layer_set_fused_local_grad(ff_layer* layer, int enable) {
  if (!layer) return FF_ERR_INVALID_ARG;
  layer->fuse_local_grad = enable != 0;
  return FF_OK;
}

ff_status ff_layer_check(ff_layer* L) {
  if (!L) return FF_ERR_INVALID_ARG;
  cudaError_t e = cudaStreamSynchronize(L->last_stream);
  if (e != cudaSuccess) return cuda_status(e, "check sync");
  int err = 0;
  FF_TRY(cudaMemcpy(&err, &L->ds->err, sizeof(int), cudaMemcpyDeviceToHost), "read error word");
  if (err) {
    const int zero = 0;
    FF_TRY(cudaMemcpy(&L->ds->err, &zero, sizeof(int), cudaMemcpyHostToDevice), "clear error word");
  }
  if (err & DEVERR_CHECK) return FF_ERR_DEVICE_CHECK;  // a skipped copy also runs waits out
  if (err & DEVERR_TIMEOUT) return FF_ERR_TIMEOUT;
  if (err & DEVERR_NONFINITE) return FF_ERR_NONFINITE;
  return FF_OK;
}

}  // extern "C"
