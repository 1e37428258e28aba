// Internal declarations shared by the libff translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "ff.h"

typedef __nv_bfloat16 bf16;

namespace ff {

// Device-side error bits latched in ff_dev_state::err.
enum : int { DEVERR_TIMEOUT = 1, DEVERR_NONFINITE = 2, DEVERR_CHECK = 4 };

// Device-side checks of the checked build (-DFF_DEVICE_CHECKS): ff_dcheck(c, err)
// is c, and latches DEVERR_CHECK in *err when c is false; in the normal build
// it is true and costs nothing.  Kernels skip the guarded access on failure.
#ifdef FF_DEVICE_CHECKS
__device__ __forceinline__ bool ff_dcheck(bool c, int* err) {
  if (!c) atomicOr(err, DEVERR_CHECK);
  return c;
}
#else
__device__ __forceinline__ bool ff_dcheck(bool, int*) { return true; }
#endif
// A tiled TMA copy must start on a 16-byte boundary of its row: the
// innermost coordinate times the element size is a multiple of 16.
__device__ __forceinline__ bool tma_x_aligned(int x, int esize) { return ((long long)x * esize) % 16 == 0; }

// Row scale and goodness helpers shared by the element-wise and GEMM kernels.
constexpr float kNormEps = 1e-12f;

// 1 / max(sqrt(ss), 1e-12), with NaN propagated (fmaxf alone would drop it).
__device__ __forceinline__ float inv_norm(float ss) {
  const float r = sqrtf(ss);
  return r != r ? r : 1.f / fmaxf(r, kNormEps);
}
// g = sum over t of gpart[t * M + i], t = 0..ntiles-1, in that order; the
// loads are issued together (8 at a time) rather than one per dependent add.
__device__ __forceinline__ float sum_partials(const float* __restrict__ gpart, int ntiles, int M, int i) {
  float g = 0.f;
  for (int t0 = 0; t0 < ntiles; t0 += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = (t0 + u < ntiles) ? __ldg(gpart + (size_t)(t0 + u) * M + i) : 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (t0 + u < ntiles) g += v[u];
  }
  return g;
}

// The FF loss terms of Eq. 1 (reading: the negative log-likelihood of the
// logistic p(real) = sigmoid(g - theta)), shared by every kernel that forms them.
__device__ __forceinline__ float softplus_f(float t) { return fmaxf(t, 0.f) + log1pf(expf(-fabsf(t))); }
__device__ __forceinline__ float sigmoid_f(float t) {
  if (t >= 0.f) return 1.f / (1.f + expf(-t));
  const float e = expf(t);
  return e / (1.f + e);
}

// Device helpers shared by the kernel files.
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Eight consecutive values of an activity row (16 bytes of bf16 or 32 of
// fp32) as floats, and back (bf16: round to nearest even).
template <typename T>
struct Vec8;
template <>
struct Vec8<bf16> {
  static __device__ __forceinline__ void load(const bf16* p, float (&v)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f = __bfloat1622float2(h[e]);
      v[2 * e] = f.x;
      v[2 * e + 1] = f.y;
    }
  }
  static __device__ __forceinline__ void store(bf16* p, const float (&v)[8]) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
    *reinterpret_cast<uint4*>(p) = u;
  }
};
template <>
struct Vec8<float> {
  static __device__ __forceinline__ void load(const float* p, float (&v)[8]) {
    const float4 a = *reinterpret_cast<const float4*>(p);
    const float4 b = *reinterpret_cast<const float4*>(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
  static __device__ __forceinline__ void store(float* p, const float (&v)[8]) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
  }
};

// One Adam step of one parameter.  a1 = lr / (1 - beta1^t) and
// r2 = 1 / (1 - beta2^t) are formed once per thread, so the update
// lr * (m / bc1) / (sqrt(v / bc2) + eps) costs one division per parameter
// instead of three (the kernel is otherwise limited by those divisions, not
// by HBM).
// Every operation is spelled out (which product is fused, every rounding),
// so all kernels that call it produce the same bits whatever the compiler's
// contraction choices at each call site.
__device__ __forceinline__ void adam1(float& w, float& m, float& v, float g, float a1, float b1, float b2, float eps,
                                      float r2) {
  m = fmaf(b1, m, __fmul_rn(1.f - b1, g));
  v = fmaf(b2, v, __fmul_rn(__fmul_rn(1.f - b2, g), g));
  w = __fsub_rn(w, __fdiv_rn(__fmul_rn(a1, m), __fadd_rn(__fsqrt_rn(__fmul_rn(v, r2)), eps)));
}

// Bound on every spin-wait in a kernel: after this many nanoseconds of
// %globaltimer the wait gives up, latches DEVERR_TIMEOUT and the kernel
// winds down.
constexpr unsigned long long kWaitTimeoutNs = 1000000000ull;  // 1 s

// Per-layer scalars that kernels read and write on the device, so that a
// captured CUDA graph replays correctly (no per-step host arguments).
struct ff_dev_state {
  long long t;        // Adam step counter (number of completed updates)
  double pow1, pow2;  // beta1^t, beta2^t
  float bc1, bc2;     // 1 - beta1^t, 1 - beta2^t of the current update
  int err;            // latched DEVERR_* bits
  float loss;         // loss of the last train step when the caller passed none
  float stats[3];     // last train step: mean g of positive rows, of negative rows, active-ReLU fraction
};

inline int row_stride(int features) { return (features + 7) & ~7; }
inline int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }

// ------------------------------------------------------------------ kernels
// All launchers return the launch status (cudaGetLastError after the launch).

// Overlay (train/forward) or label-area zeroing (predict), cast, row scale.
//   mode 0: out[:,0..9] = one-hot(labels[r]); mode 1: out[:,0..9] = 0 and the
//   norm counts one extra 1.0 (the one-hot every predict overlay adds);
//   mode 2: out[:,0..9] = 0.1, the neutral label of the softmax head (§3).
// Output row r reads input row r % src_rows (src_rows 0: rows): with
// src_rows = B the B images of a pair batch are read once each for both
// their positive and their negative row.
cudaError_t launch_overlay(const float* x, const int* labels, int rows, int F, void* out,
                           int ldo, bool out_bf16, float* s_out, int mode, cudaStream_t st, int src_rows = 0);
// s_r = 1 / max(||x_r||, 1e-12) of an activation buffer.
cudaError_t launch_row_scale(const void* x, int ldx, bool x_bf16, int rows, int F,
                             float* s_out, cudaStream_t st);
// Goodness from the forward GEMM's per-tile partials (forward and predict).
struct FinalizeArgs {
  const float* gpart; int ntiles; int M;
  float* g_out;        // [M] or null
  float* s_next;       // [M] or null
  float* G_acc;        // [M] predict goodness accumulator or null
  int* err;            // error word
};
int finalize_grid(int M);
cudaError_t launch_finalize(const FinalizeArgs& a, cudaStream_t st);
// Train step after the forward GEMM: goodness, loss, dL/dg, next-layer scale,
// dZ' = (s * 2 dL/dg) * H in the operand type, db partials per 32 rows, and
// the Adam step counter / bias-correction terms.
struct GradPrepArgs {
  const float* gpart; int ntiles; int M; int N; int ld;  // ld: row stride of H and dZ
  int B; float theta;
  const float* s;      // [M] row scale of this layer's input
  float* g_out;        // [M] or null
  float* s_next;       // [M] or null
  float* dbpart;       // [row blocks, N]
  float* loss_part;    // [row blocks]; the Adam kernel reduces them into the loss
  float* stat_part;    // [2 * row blocks + row blocks * ncb]: g sums of positive / negative rows, active counts
  int ncb;             // column blocks (256 columns each)
  ff_dev_state* ds;
  double beta1, beta2;
  int* err;
};
cudaError_t launch_grad_prep(const GradPrepArgs& a, bool b16, const void* H, void* dZ, cudaStream_t st);
int local_grad_row_blocks(int M);
struct AdamArgs {
  float* W; float* mW; float* vW; const float* dW; int N; int K;
  bf16* Wb; int ldb;      // bf16 copy of W or null
  float* b; float* mb; float* vb; const float* dbpart; int nrb; float* db_out;
  int has_bias;
  float lr, beta1, beta2, eps;
  const ff_dev_state* ds;
  const float* loss_part;  // [nrb] grad_prep's loss partials of this step, or null
  float* loss_out;         // [1] receives their sum / B
  int B;
  const float* stat_part;  // grad_prep's statistics partials, or null
  int ncb;
  float* stats_out;        // [3] receives the step's statistics
  // Dead data: buffers (128-byte aligned, whole lines) that nothing reads
  // before they are rewritten, and dW itself once read (discard_dW), have
  // their lines dropped from L2 instead of written back to HBM.
  int discard_dW;
  int ndead;
  char* dead[2];
  long long dead_lines[2];
};
// Adds [p, p + bytes) to the Adam step's dead buffers (its whole 128-byte
// lines; nothing when p is not 128-byte aligned).
void add_dead(AdamArgs& a, void* p, size_t bytes);

// Launch configuration with programmatic stream serialization: the kernel
// may start while the previous kernel of the stream finishes and waits for it
// with griddep_wait() before touching memory.
struct PdlLaunch {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  PdlLaunch(dim3 grid, dim3 block, cudaStream_t st, size_t smem = 0) {
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
  }
};

cudaError_t launch_adam(const AdamArgs& a, cudaStream_t st);
cudaError_t launch_init_weights(float* W, int N, int K, unsigned long long seed, cudaStream_t st);
cudaError_t launch_to_bf16(const float* W, int N, int K, bf16* Wb, int ldb, cudaStream_t st);
// predict helpers
cudaError_t launch_label_columns(const void* W, int ldw, bool w_bf16, int N, float* cols /*[10,ldc]*/,
                                 int ldc, cudaStream_t st);
cudaError_t launch_expand(const float* base, int ldbase, const float* cols, const float* s1,
                          const float* bias, int n, int N, void* H, int ldh, bool h_bf16,
                          float* s_next, float* G_acc /*null unless single layer*/, int* err,
                          cudaStream_t st);
cudaError_t launch_argmax(const float* G, int n, const int* labels, int* pred, cudaStream_t st);
// one bounded wait on an mbarrier nothing arrives on (latches DEVERR_TIMEOUT)
cudaError_t launch_wait_selftest(int* err, unsigned long long timeout_ns, cudaStream_t st);

// ------------------------------------------------------------------- GEMMs
// Forward epilogue: H = ReLU(s_r * acc + b) (bf16 or fp32), per-tile goodness
// partials gpart[tile_n * M + r].  Store epilogue: C = acc (fp32).
struct EpiArgs {
  const float* row_scale;
  const float* bias;   // null: no bias
  void* out; int ldo;
  float* gpart;        // forward only
  // Forward GEMMs of the tensor-core path only: with gpart_in set, the row
  // scale is inv_norm of the previous layer's goodness (its partials
  // gpart_in[t * M + i], t < ntiles_in, summed as k_finalize does) instead of
  // row_scale[i]; the first column tile adds that goodness to G_acc[i] and
  // stores the scale in s_out[i] (each when set) and flags a non-finite one.
  const float* gpart_in;
  int ntiles_in;
  float* G_acc;
  float* s_out;
  // fp32 SIMT GEMMs only: split-K scratch (partial tiles, capacity in floats,
  // and one arrival counter per output tile, zero between launches); null: no
  // split.
  float* kpart;
  size_t kpart_cap;
  int* kcnt;
  int kcnt_cap;
  // Tensor-core forward GEMMs: a grid that would fill at most half the SMs
  // may use 128-column tiles (twice the CTAs).  Set where the GEMM has the
  // GPU to itself (the layer chains of predict and of the softmax head); the
  // net's concurrent per-layer GEMMs run faster on the wider tiles.
  bool narrow;
  // Tensor-core forward GEMMs: with logit_V set ([10, logit_ldV] fp32, the
  // weights of a 10-class softmax block on this layer's activity), each
  // epilogue warp also writes its rows' partial logits over its columns,
  // zpart[(t * M + i) * 10 + c] = sum over the columns j of tile-half t of
  // bf16(H_ij) V_cj, with t indexing like the goodness partials.
  const float* logit_V;
  int logit_ldV;
  float* zpart;
};

// Tensor-core (tcgen05) bf16 GEMMs, fp32 accumulate.
//   fwd/store: C[M,N] = A[M,K] B[N,K]^T  (A, B row-major, K contiguous)
//   wgrad:     C[N,K] = G[R,N]^T X[R,K]  (contraction over R rows)
// Goodness partials per row the forward GEMM writes for an M x N output (its
// tile shape depends on both and on EpiArgs::narrow), and the most it writes
// for any M.
int tc_fwd_ntiles(int M, int N, bool narrow);
int tc_fwd_ntiles_max(int N);
cudaError_t tc_gemm_fwd(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K,
                        const EpiArgs& ep, int* err, cudaStream_t st);
// The train step's forward with the local step fused into its epilogue: the
// forward above (H into ep.out) and everything the local-gradient kernel
// (launch_grad_prep) computes from it -- dZ' into dZ ([M, ep.ldo] bf16), the
// bias-gradient, loss and statistics partials, g_out, s_next and the Adam
// step counter of lg -- bitwise the same.  lg.gpart and lg.ntiles are not
// used; ep.row_scale must be lg.s.  For N <= 2048 where the GPU can hold the
// clusters (tc_fwd_lg_supported); cudaErrorInvalidValue otherwise.
bool tc_fwd_lg_supported(int M, int N);
cudaError_t tc_gemm_fwd_lg(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                           const GradPrepArgs& lg, bf16* dZ, int* err, cudaStream_t st);
cudaError_t tc_gemm_store(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K,
                          float* C, int ldc, int* err, cudaStream_t st);
// The same forward (without gpart_in or block logits) and store GEMMs on fp32
// operands, as three TF32 tensor-core products per term (Ah Bh + Ah Bl +
// Al Bh; relative error near 2^-21 per product); H is written in fp32.  For K
// and both row strides multiples of 4 (tc_f32_supported).
bool tc_f32_supported(int K, int lda, int ldb);
cudaError_t tc_gemm_fwd_f32(const float* A, int lda, const float* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                            int* err, cudaStream_t st);
cudaError_t tc_gemm_store_f32(const float* A, int lda, const float* B, int ldb, int M, int N, int K, float* C, int ldc,
                              int* err, cudaStream_t st);
cudaError_t tc_gemm_wgrad(const bf16* G, int ldg, const bf16* X, int ldx, int R, int N, int K,
                          float* C, int ldc, int* err, cudaStream_t st);
bool tc_supported();
// CTAs of the forward GEMM for an M x N output (its tile configuration).
int tc_gemm_fwd_ctas(int M, int N, bool narrow);
// Tensor map of a row-major [rows, cols] bf16 (esize 2) or fp32 (esize 4)
// matrix with row stride ld, boxes of box_rows x box_cols, no swizzle; false
// if the pointer or the stride is not 16-byte aligned.
bool make_plain_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols,
                    int box_rows);
// The same with 128-byte swizzle (the layout the tensor-core GEMMs' shared
// memory descriptors expect); out-of-range elements of a box read as zero.
bool make_sw128_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols,
                    int box_rows);

// SIMT fp32 GEMMs with the same contracts.  A GEMM of few output tiles
// splits its contraction over blockIdx.z when the EpiArgs carry split-K
// scratch of the size simt_split_floats / simt_split_tiles give (the wgrad
// form takes the scratch from `split`).
int simt_fwd_ntiles(int N);
size_t simt_split_floats(int M, int N, int K);
int simt_split_tiles(int M, int N);
cudaError_t simt_gemm_fwd(const float* A, int lda, const float* B, int ldb, int M, int N, int K,
                          const EpiArgs& ep, cudaStream_t st);
cudaError_t simt_gemm_store(const float* A, int lda, const float* B, int ldb, int M, int N, int K,
                            float* C, int ldc, cudaStream_t st);
cudaError_t simt_gemm_wgrad(const float* G, int ldg, const float* X, int ldx, int R, int N, int K,
                            float* C, int ldc, cudaStream_t st, const EpiArgs* split = nullptr);

}  // namespace ff

// The layer object behind the opaque handle.
struct ff_layer {
  ff_layer_config cfg;
  int K, N, ldK, ldN;
  int device;
  bool is_bf16;
  cudaStream_t last_stream;
  // parameters and Adam moments (fp32, dense [N,K] / [N])
  float *W, *b, *mW, *vW, *mb, *vb;
  bf16* Wb;          // [N, ldK] bf16 copy (bf16 mode)
  float* db;         // [N] reduced bias gradient of the last step
  float* dW;         // [N, K] weight gradient of the last step
  ff::ff_dev_state* ds;
  // workspace, capacity cap rows
  int cap;
  void* X;           // [cap, ldK] overlay output
  float* s_in;       // [cap]
  void* H;           // [cap, ldN] activity when the caller passes no h_out
  void* dZ;          // [cap, ldN] weight-gradient operand s*dZ
  float* gpart;      // [ntiles, cap]
  float* g;          // [cap]
  float* c;          // [cap]
  float* s_next;     // [cap]
  float* dbpart;     // [row blocks, N]
  float* loss_part;  // [max(finalize blocks, row blocks)]
  float* stat_part;  // [row blocks * (2 + column blocks)] step statistics partials
  // predict scratch (owned here when this layer is layers[0] of ff_predict)
  void* pws; size_t pws_bytes;
  // split-K scratch of the fp32 GEMMs (grown on demand; counters kept zero)
  float* kpart; size_t kpart_cap;
  int* kcnt; int kcnt_cap;
  // bf16 train steps: the local gradient in the forward GEMM's epilogue
  // (tc_gemm_fwd_lg) where the shape allows, else the separate kernel.  Off
  // by default: on the 784-2000x4 epoch with 4 layer streams the fused
  // forward made the epoch slower (9.0 against 8.1 ms): its 8-CTA clusters
  // wait for 8 free SMs of one GPC while the other layers' kernels run, and
  // its longer epilogue holds them, where the separate kernel fills gaps on
  // every SM; alone on one stream it is 2 % faster than forward + kernel.
  bool fuse_local_grad = false;
};
