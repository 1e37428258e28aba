// Bandwidth-bound kernels of the FF layer step and of goodness prediction:
//   overlay      §3 "Negative Data": one-hot label in features 0..9, cast to
//                the operand type, row norm for x / max(||x||, 1e-12)
//   finalize     Eq. 1: goodness from the GEMM's per-tile partials and the
//                next layer's row scale (forward and predict)
//   grad_prep    the same goodness, the pair loss softplus(theta - g_pos) +
//                softplus(g_neg - theta) and its derivative dL/dg, then
//                dZ = dL/dg * 2h (h = 0 where z <= 0), the weight-gradient
//                operand s*dZ and per-32-row partial sums for db
//   adam         Adam (§5.1) on W and b, refreshing the bf16 copy of W, and
//                dropping the step's dead data (dW, s*dZ) from L2
//   init         He-uniform W from a counter-based SplitMix64 stream
//   predict      label columns of W1, per-label expansion of layer 1,
//                argmax over the 10 labels (§3 "Prediction"), and over
//                the 9 wrong labels for AdaptiveNEG negatives (§5)
// Reductions use fixed orders (no floating-point atomics), so results do not
// depend on scheduling.
#include "ff_internal.cuh"
#include "ff_ptx.cuh"

namespace ff {
namespace {

// ReLU that keeps NaN visible to the non-finite check.
__device__ __forceinline__ float relu_nan(float z) { return z != z ? z : fmaxf(z, 0.f); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }
__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }

// ------------------------------------------------------------------ overlay
template <typename T>
__device__ __forceinline__ void store4(T* p, float a, float b, float c, float d);
template <>
__device__ __forceinline__ void store4<float>(float* p, float a, float b, float c, float d) {
  *reinterpret_cast<float4*>(p) = make_float4(a, b, c, d);
}
template <>
__device__ __forceinline__ void store4<bf16>(bf16* p, float a, float b, float c, float d) {
  __nv_bfloat162 p0 = __floats2bfloat162_rn(a, b), p1 = __floats2bfloat162_rn(c, d);
  *reinterpret_cast<uint2*>(p) = make_uint2(*reinterpret_cast<uint32_t*>(&p0), *reinterpret_cast<uint32_t*>(&p1));
}

// One warp per row.  Rows whose length is a multiple of 4 (16-byte aligned
// when x is) move as float4; others element by element.
template <typename T>
__global__ void k_overlay(const float* __restrict__ x, const int* __restrict__ labels, int rows, int F,
                          T* __restrict__ out, int ldo, float* __restrict__ s_out, int mode, int src_rows) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + warp;
  if (row >= rows) return;
  const float* xr = x + (size_t)(row % src_rows) * F;
  T* orow = out + (size_t)row * ldo;
  const int lab = (mode == 0 && labels) ? labels[row] : -1;
  float ss = 0.f;
  const bool vec = (F & 3) == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  if (vec) {
    for (int f = 4 * lane; f < ldo; f += 128) {
      float v[4] = {0.f, 0.f, 0.f, 0.f};
      if (f < F) {
        const float4 q = __ldg(reinterpret_cast<const float4*>(xr + f));
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (f + u < 10) v[u] = mode == 2 ? 0.1f : (f + u == lab) ? 1.f : 0.f;
        ss = fmaf(v[u], v[u], ss);
      }
      store4<T>(orow + f, v[0], v[1], v[2], v[3]);
    }
  } else {
    for (int f = lane; f < ldo; f += 32) {
      float v = 0.f;
      if (f < F) v = (f < 10) ? (mode == 2 ? 0.1f : f == lab ? 1.f : 0.f) : __ldg(xr + f);
      orow[f] = from_f<T>(v);
      ss = fmaf(v, v, ss);
    }
  }
  ss = warp_sum(ss);
  if (lane == 0 && s_out) s_out[row] = inv_norm(ss + (mode == 1 ? 1.f : 0.f));
}

template <typename T>
__global__ void k_row_scale(const T* __restrict__ x, int ldx, int rows, int F, float* __restrict__ s_out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + warp;
  if (row >= rows) return;
  const T* xr = x + (size_t)row * ldx;
  float ss = 0.f;
  for (int f = lane; f < F; f += 32) {
    const float v = to_f(xr[f]);
    ss = fmaf(v, v, ss);
  }
  ss = warp_sum(ss);
  if (lane == 0) s_out[row] = inv_norm(ss);
}

// ----------------------------------------------------------------- finalize

__global__ void __launch_bounds__(256) k_finalize(FinalizeArgs a) {
  ptx::griddep_wait();  // launched with programmatic stream serialization
  const int i = blockIdx.x * 256 + threadIdx.x;
  if (i >= a.M) return;
  const float g = sum_partials(a.gpart, a.ntiles, a.M, i);
  if (!isfinite(g)) atomicOr(a.err, DEVERR_NONFINITE);
  if (a.g_out) a.g_out[i] = g;
  if (a.s_next) a.s_next[i] = inv_norm(g);
  if (a.G_acc) a.G_acc[i] += g;
}

// --------------------------------------------------------------- local grad
// Train-step epilogue of the forward GEMM, one block per 32 rows x 256
// columns (block 32 x 8).  Thread (x, y) owns columns 8x..8x+7 of rows
// y, y+8, y+16, y+24: it issues those activity loads first; meanwhile the
// warp's lanes, 8 per row, reduce the per-tile goodness partials of its four
// rows and lanes 0, 8, 16, 24 form dL/dg, broadcast to the warp by shuffles.
// Then
//   dZ'_ij = s_i * 2 dL/dg_i * h_ij (h = 0 where z <= 0) in the operand type,
//   and the block's column sums of dZ for db.
// Blocks of column 0 also write g, the next layer's scale
// 1/max(sqrt g, 1e-12) and the block's loss partial (reduced by the Adam
// kernel that follows on the same stream); block (0, 0) advances the Adam
// step t and its bias-correction terms.
constexpr int kGradRows = 32;

template <typename T>
__global__ void __launch_bounds__(256) k_grad_prep(GradPrepArgs a, const T* __restrict__ H, T* __restrict__ dZ) {
  ptx::griddep_wait();  // launched with programmatic stream serialization
  __shared__ float red[8][256 + 8];
  __shared__ float lred[8], gpred[8], gnred[8], ared[8];
  const int r0 = blockIdx.y * kGradRows;
  const bool lead = blockIdx.x == 0;
  const int lane = threadIdx.x;
  const int cg = blockIdx.x * 256 + lane * 8;
  const bool cols_ok = cg < a.ld;
  float h[4][8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int i = r0 + threadIdx.y + 8 * k;
    if (cols_ok && i < a.M) {
      Vec8<T>::load(H + (size_t)i * a.ld + cg, h[k]);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) h[k][e] = 0.f;
    }
  }
  // The warp's 4 rows r0 + y + 8k: lanes 8k .. 8k+7 share row k's goodness,
  // lane 8k + p loading partials p, p + 8, ... (one round trip for up to 64
  // column-tile partials) and a fixed xor tree adding the 8 lane sums; lane 8k
  // then forms the row's loss terms.
  float cc = 0.f, sc = 0.f, lv = 0.f, gp = 0.f, gn = 0.f;
  {
    const int k = lane >> 3, p = lane & 7;
    const int i = r0 + threadIdx.y + 8 * k;
    float g = 0.f;
    if (i < a.M) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int t = p + 8 * u;
        v[u] = t < a.ntiles ? __ldg(a.gpart + (size_t)t * a.M + i) : 0.f;
      }
      for (int t = p + 64; t < a.ntiles; t += 8) v[0] += __ldg(a.gpart + (size_t)t * a.M + i);  // past 64 tiles
#pragma unroll
      for (int u = 0; u < 8; ++u) g += v[u];
    }
    g += __shfl_xor_sync(0xffffffffu, g, 4);
    g += __shfl_xor_sync(0xffffffffu, g, 2);
    g += __shfl_xor_sync(0xffffffffu, g, 1);
    if (p == 0 && i < a.M) {
      const bool pos = i < a.B;
      const float tt = pos ? a.theta - g : g - a.theta;  // the pair member's margin error
      const float sg = sigmoid_f(tt);
      cc = 2.f * (pos ? -sg : sg) / (float)a.B;
      sc = a.s[i] * cc;
      if (lead) {
        if (!isfinite(g)) atomicOr(a.err, DEVERR_NONFINITE);
        if (a.g_out) a.g_out[i] = g;
        if (a.s_next) a.s_next[i] = inv_norm(g);
        lv = softplus_f(tt);
        (pos ? gp : gn) = g;
      }
    }
  }
  float db[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) db[e] = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float ck = __shfl_sync(0xffffffffu, cc, 8 * k), sk = __shfl_sync(0xffffffffu, sc, 8 * k);
    const int i = r0 + threadIdx.y + 8 * k;
    float z[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      z[e] = sk * h[k][e];
      db[e] = fmaf(ck, h[k][e], db[e]);
    }
    if (cols_ok && i < a.M) Vec8<T>::store(dZ + (size_t)i * a.ld + cg, z);
  }
  if (lead) {
    lv = warp_sum(lv);  // only lanes 0, 8, 16, 24 contribute
    gp = warp_sum(gp);
    gn = warp_sum(gn);
    if (lane == 0) {
      lred[threadIdx.y] = lv;
      gpred[threadIdx.y] = gp;
      gnred[threadIdx.y] = gn;
    }
  }
  if (a.stat_part) {
    // active ReLUs among this thread's values (zero past the rows and columns)
    float act = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k)
#pragma unroll
      for (int e = 0; e < 8; ++e) act += h[k][e] > 0.f ? 1.f : 0.f;
    act = warp_sum(act);
    if (lane == 0) ared[threadIdx.y] = act;
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) red[threadIdx.y][lane * 8 + e] = db[e];
  __syncthreads();
  if (threadIdx.y == 0) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int j = cg + e;
      float t = 0.f;
#pragma unroll
      for (int y = 0; y < 8; ++y) t += red[y][lane * 8 + e];
      if (j < a.N) a.dbpart[(size_t)blockIdx.y * a.N + j] = t;
    }
    if (a.stat_part && lane == 0) {
      float t = 0.f;
#pragma unroll
      for (int y = 0; y < 8; ++y) t += ared[y];
      a.stat_part[2 * gridDim.y + (size_t)blockIdx.y * a.ncb + blockIdx.x] = t;
    }
    if (lead && lane == 0) {
      float t = 0.f;
#pragma unroll
      for (int y = 0; y < 8; ++y) t += lred[y];
      a.loss_part[blockIdx.y] = t;
      if (a.stat_part) {
        float tp = 0.f, tn = 0.f;
#pragma unroll
        for (int y = 0; y < 8; ++y) {
          tp += gpred[y];
          tn += gnred[y];
        }
        a.stat_part[blockIdx.y] = tp;
        a.stat_part[gridDim.y + blockIdx.y] = tn;
      }
    }
    if (lead && blockIdx.y == 0 && lane == 0) {
      // the Adam update that follows is step t; beta^t kept as running products
      a.ds->t += 1;
      a.ds->pow1 *= a.beta1;
      a.ds->pow2 *= a.beta2;
      a.ds->bc1 = (float)(1.0 - a.ds->pow1);
      a.ds->bc2 = (float)(1.0 - a.ds->pow2);
    }
  }
}

// --------------------------------------------------------------------- Adam
// W, m, v (float4 when K % 4 == 0) through adam1 (ff_internal.cuh); the bias
// elements, db from grad_prep's partials, and the step's loss and statistics
// in the blocks past w_blocks.
__global__ void __launch_bounds__(256) k_adam(AdamArgs a, int w_blocks) {
  ptx::griddep_wait();  // launched with programmatic stream serialization
  {
    // the step's dead buffers: every kernel that reads them has completed
    const long long gt = (long long)blockIdx.x * 256 + threadIdx.x, nt = (long long)gridDim.x * 256;
    for (int r = 0; r < a.ndead; ++r)
      for (long long l = gt; l < a.dead_lines[r]; l += nt) ptx::discard_l2(a.dead[r] + l * 128);
  }
  const float a1 = a.lr / a.ds->bc1, r2 = 1.f / a.ds->bc2;
  if ((int)blockIdx.x < w_blocks) {
    const long long total = (long long)a.N * a.K;
    const long long stride = (long long)w_blocks * 256;
    if ((a.K & 3) == 0) {
      // bf16 copy addressed like W when its rows are not padded
      const bool dense_b = a.ldb == a.K;
      for (long long q = (long long)blockIdx.x * 256 + threadIdx.x; q * 4 < total; q += stride) {
        const long long idx = q * 4;
        // W, m, v and dW are touched once per step: evict-first, so the
        // stream leaves the GEMMs' operands in L2
        float4 w = __ldcs(reinterpret_cast<const float4*>(a.W + idx));
        float4 m = __ldcs(reinterpret_cast<const float4*>(a.mW + idx));
        float4 v = __ldcs(reinterpret_cast<const float4*>(a.vW + idx));
        const float4 g = __ldcs(reinterpret_cast<const float4*>(a.dW + idx));
        adam1(w.x, m.x, v.x, g.x, a1, a.beta1, a.beta2, a.eps, r2);
        adam1(w.y, m.y, v.y, g.y, a1, a.beta1, a.beta2, a.eps, r2);
        adam1(w.z, m.z, v.z, g.z, a1, a.beta1, a.beta2, a.eps, r2);
        adam1(w.w, m.w, v.w, g.w, a1, a.beta1, a.beta2, a.eps, r2);
        __stcs(reinterpret_cast<float4*>(a.W + idx), w);
        __stcs(reinterpret_cast<float4*>(a.mW + idx), m);
        __stcs(reinterpret_cast<float4*>(a.vW + idx), v);
        // the first of every 8 threads drops the 128-byte dW line the 8 just
        // read (the warp's loads have all returned: g was used above)
        if (a.discard_dW && (threadIdx.x & 7) == 0 && idx + 32 <= total) ptx::discard_l2(a.dW + idx);
        if (a.Wb) {
          const long long o = dense_b ? idx : (idx / a.K) * a.ldb + idx % a.K;
          __nv_bfloat162 p0 = __floats2bfloat162_rn(w.x, w.y), p1 = __floats2bfloat162_rn(w.z, w.w);
          uint2 u = make_uint2(*reinterpret_cast<uint32_t*>(&p0), *reinterpret_cast<uint32_t*>(&p1));
          *reinterpret_cast<uint2*>(a.Wb + o) = u;
        }
      }
    } else {
      for (long long idx = (long long)blockIdx.x * 256 + threadIdx.x; idx < total; idx += stride) {
        float w = a.W[idx], m = a.mW[idx], v = a.vW[idx];
        adam1(w, m, v, a.dW[idx], a1, a.beta1, a.beta2, a.eps, r2);
        a.W[idx] = w;
        a.mW[idx] = m;
        a.vW[idx] = v;
        if (a.Wb) a.Wb[(idx / a.K) * a.ldb + idx % a.K] = __float2bfloat16_rn(w);
      }
    }
  } else {
    // 32 bias elements per block: warp w sums row blocks w, w+8, ... for the
    // block's 32 columns (lane = column), then warp 0 adds the 8 warp sums in
    // order -- a fixed reduction order, with the loads batched.
    __shared__ float part[8][33];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int j = (blockIdx.x - w_blocks) * 32 + lane;
    float acc = 0.f;
    if (j < a.N) {
      for (int rb0 = w; rb0 < a.nrb; rb0 += 64) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int rb = rb0 + 8 * u;
          v[u] = rb < a.nrb ? __ldg(a.dbpart + (size_t)rb * a.N + j) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) acc += v[u];
      }
    }
    part[w][lane] = acc;
    __syncthreads();
    if (blockIdx.x == w_blocks && w == 1 && a.loss_part) {
      // the step's loss: grad_prep's per-row-block partials, lane-strided then
      // a fixed-order warp tree
      float tot = 0.f;
      for (int rb = lane; rb < a.nrb; rb += 32) tot += a.loss_part[rb];
      tot = warp_sum(tot);
      if (lane == 0) a.loss_out[0] = tot / (float)a.B;
    }
    if (blockIdx.x == w_blocks && w >= 2 && w <= 4 && a.stat_part) {
      // the step's statistics: mean goodness of the positive and of the
      // negative rows, and the fraction of active ReLUs
      const int n = w == 4 ? a.nrb * a.ncb : a.nrb;
      const float* src = a.stat_part + (w == 2 ? 0 : w == 3 ? a.nrb : 2 * a.nrb);
      float tot = 0.f;
      for (int k = lane; k < n; k += 32) tot += src[k];
      tot = warp_sum(tot);
      if (lane == 0) a.stats_out[w - 2] = w == 4 ? tot / (2.f * (float)a.B * (float)a.N) : tot / (float)a.B;
    }
    if (w != 0 || j >= a.N) return;
    float db = 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u) db += part[u][lane];
    if (a.db_out) a.db_out[j] = db;
    if (a.has_bias) {
      float b = a.b[j], m = a.mb[j], v = a.vb[j];
      adam1(b, m, v, db, a1, a.beta1, a.beta2, a.eps, r2);
      a.b[j] = b;
      a.mb[j] = m;
      a.vb[j] = v;
    }
  }
}

// --------------------------------------------------------------------- init
// SplitMix64 (Steele, Lea, Flood 2014; finaliser constants of Vigna's
// splitmix64.c), used counter-based: output i of a stream with initial
// state s0 is mix(s0 + (i + 1) * gamma).
__device__ __host__ __forceinline__ unsigned long long sm64_mix(unsigned long long z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
constexpr unsigned long long kGamma = 0x9E3779B97F4A7C15ull;
constexpr unsigned long long kStreamWeights = 4;

__global__ void k_init_weights(float* __restrict__ W, long long total, unsigned long long s0, double bound) {
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const unsigned long long r = sm64_mix(s0 + (unsigned long long)(i + 1) * kGamma);
    const double u = (double)(r >> 11) * 0x1.0p-53;
    W[i] = (float)((2.0 * u - 1.0) * bound);
  }
}

__global__ void k_to_bf16(const float* __restrict__ W, int N, int K, bf16* __restrict__ Wb, int ldb) {
  const long long total = (long long)N * ldb;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    const long long n = i / ldb, k = i % ldb;
    Wb[i] = __float2bfloat16_rn(k < K ? W[n * K + k] : 0.f);
  }
}

// ------------------------------------------------------------------ predict
template <typename T>
__global__ void k_label_columns(const T* __restrict__ W, int ldw, int N, float* __restrict__ cols, int ldc) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= ldc) return;
#pragma unroll
  for (int c = 0; c < 10; ++c) cols[(size_t)c * ldc + j] = j < N ? to_f(W[(size_t)j * ldw + c]) : 0.f;
}

// One block per sample: for each label c the layer-1 activity of the
// overlaid input, h = ReLU(s * (base + W[:, c]) + b), using
//   overlay(x, c) W^T = x0 W^T + W[:, c]   (x0: x with features 0..9 zeroed)
// and the goodness/next scale of that row (row r = 10 * sample + c).  Each
// thread takes 8 consecutive columns: the base row and the bias are read
// once for all 10 labels, the 10 goodness sums stay in registers and are
// reduced once at the end (warp, then the 8 warps in order).
template <typename T>
__global__ void __launch_bounds__(256) k_expand(const float* __restrict__ base, int ldbase,
                                                const float* __restrict__ cols, const float* __restrict__ s1,
                                                const float* __restrict__ bias, int N, T* __restrict__ H, int ldh,
                                                float* __restrict__ s_next, float* __restrict__ G_acc, int* err) {
  __shared__ float red[8][10];
  const int n = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float s = s1[n];
  const float* brow = base + (size_t)n * ldbase;
  float g[10];
#pragma unroll
  for (int c = 0; c < 10; ++c) g[c] = 0.f;
  for (int j = 8 * threadIdx.x; j < ldh; j += 8 * 256) {
    float b8[8], bi[8];
    const float4 p = *reinterpret_cast<const float4*>(brow + j);
    const float4 q = *reinterpret_cast<const float4*>(brow + j + 4);
    b8[0] = p.x; b8[1] = p.y; b8[2] = p.z; b8[3] = p.w;
    b8[4] = q.x; b8[5] = q.y; b8[6] = q.z; b8[7] = q.w;
#pragma unroll
    for (int e = 0; e < 8; ++e) bi[e] = (bias && j + e < N) ? __ldg(bias + j + e) : 0.f;
#pragma unroll
    for (int c = 0; c < 10; ++c) {
      const float* cr = cols + (size_t)c * ldh + j;
      const float4 u = __ldg(reinterpret_cast<const float4*>(cr));
      const float4 v = __ldg(reinterpret_cast<const float4*>(cr + 4));
      const float cv[8] = {u.x, u.y, u.z, u.w, v.x, v.y, v.z, v.w};
      float h[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        float z = s * (b8[e] + cv[e]);
        if (bias) z += bi[e];
        h[e] = j + e < N ? relu_nan(z) : 0.f;
        g[c] = fmaf(h[e], h[e], g[c]);
      }
      Vec8<T>::store(H + ((size_t)n * 10 + c) * ldh + j, h);
    }
  }
#pragma unroll
  for (int c = 0; c < 10; ++c) {
    const float v = warp_sum(g[c]);
    if (lane == 0) red[warp][c] = v;
  }
  __syncthreads();
  if (threadIdx.x < 10) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += red[w][threadIdx.x];
    const size_t r = (size_t)n * 10 + threadIdx.x;
    if (!isfinite(t)) atomicOr(err, DEVERR_NONFINITE);
    s_next[r] = inv_norm(t);
    if (G_acc) G_acc[r] += t;
  }
}

// pred[i] = the label with the largest G[i, c], the lowest on ties.  With
// labels (AdaptiveNEG, §5) the sample's own label is left out, so pred[i] is
// its strongest wrong label; a label outside 0..9 leaves nothing out.
__global__ void k_argmax(const float* __restrict__ G, int n, const int* __restrict__ labels,
                         int* __restrict__ pred) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float* g = G + (size_t)i * 10;
  const int skip = labels ? labels[i] : -1;
  int best = -1;
  float bv = 0.f;
#pragma unroll
  for (int c = 0; c < 10; ++c) {
    if (c == skip) continue;
    const float v = g[c];
    if (best < 0 || v > bv) {
      bv = v;
      best = c;
    }
  }
  pred[i] = best;
}

// Self-test of the bounded waits: one thread waits on an mbarrier that
// nothing arrives on, through the same bounded wait the GEMMs use, and
// latches DEVERR_TIMEOUT when it gives up.
__global__ void k_wait_selftest(int* err, unsigned long long timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    ptx::mbar_init(&bar, 1);
    abort_flag = 0;
    ptx::fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !ptx::mbar_wait(&bar, 0, timeout_ns, &abort_flag)) atomicOr(err, DEVERR_TIMEOUT);
}

int grid_for(long long work, int per_block, int cap) {
  long long b = (work + per_block - 1) / per_block;
  if (b < 1) b = 1;
  return (int)(b > cap ? cap : b);
}

}  // namespace

cudaError_t launch_overlay(const float* x, const int* labels, int rows, int F, void* out, int ldo, bool out_bf16,
                           float* s_out, int mode, cudaStream_t st, int src_rows) {
  if (rows <= 0) return cudaSuccess;
  if (src_rows <= 0 || src_rows > rows) src_rows = rows;
  const int grid = cdiv(rows, 8);
  if (out_bf16)
    k_overlay<bf16><<<grid, 256, 0, st>>>(x, labels, rows, F, (bf16*)out, ldo, s_out, mode, src_rows);
  else
    k_overlay<float><<<grid, 256, 0, st>>>(x, labels, rows, F, (float*)out, ldo, s_out, mode, src_rows);
  return cudaGetLastError();
}

cudaError_t launch_row_scale(const void* x, int ldx, bool x_bf16, int rows, int F, float* s_out, cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  const int grid = cdiv(rows, 8);
  if (x_bf16)
    k_row_scale<bf16><<<grid, 256, 0, st>>>((const bf16*)x, ldx, rows, F, s_out);
  else
    k_row_scale<float><<<grid, 256, 0, st>>>((const float*)x, ldx, rows, F, s_out);
  return cudaGetLastError();
}

int finalize_grid(int M) { return cdiv(M, 256); }

cudaError_t launch_finalize(const FinalizeArgs& a, cudaStream_t st) {
  if (a.M <= 0) return cudaSuccess;
  PdlLaunch l(dim3(finalize_grid(a.M)), dim3(256), st);
  return cudaLaunchKernelEx(&l.cfg, k_finalize, a);
}

int local_grad_row_blocks(int M) { return cdiv(M, kGradRows); }

cudaError_t launch_grad_prep(const GradPrepArgs& a, bool b16, const void* H, void* dZ, cudaStream_t st) {
  PdlLaunch l(dim3(cdiv(a.ld, 256), local_grad_row_blocks(a.M)), dim3(32, 8), st);
  if (b16) return cudaLaunchKernelEx(&l.cfg, k_grad_prep<bf16>, a, (const bf16*)H, (bf16*)dZ);
  return cudaLaunchKernelEx(&l.cfg, k_grad_prep<float>, a, (const float*)H, (float*)dZ);
}

void add_dead(AdamArgs& a, void* p, size_t bytes) {
  if (!p || ((uintptr_t)p & 127u) || bytes < 128 || a.ndead >= 2) return;
  a.dead[a.ndead] = static_cast<char*>(p);
  a.dead_lines[a.ndead] = (long long)(bytes / 128);
  ++a.ndead;
}

cudaError_t launch_adam(const AdamArgs& a, cudaStream_t st) {
  const long long total = (long long)a.N * a.K;
  const int w_blocks = grid_for((a.K & 3) == 0 ? total / 4 : total, 256, 152 * 16);
  const int b_blocks = cdiv(a.N, 32);
  PdlLaunch l(dim3(w_blocks + b_blocks), dim3(256), st);
  return cudaLaunchKernelEx(&l.cfg, k_adam, a, w_blocks);
}

cudaError_t launch_init_weights(float* W, int N, int K, unsigned long long seed, cudaStream_t st) {
  const long long total = (long long)N * K;
  const unsigned long long key = ((seed & ((1ull << 56) - 1)) << 8) | kStreamWeights;
  const unsigned long long s0 = sm64_mix(key);
  const double bound = std::sqrt(6.0 / (double)K);
  k_init_weights<<<grid_for(total, 256, 152 * 32), 256, 0, st>>>(W, total, s0, bound);
  return cudaGetLastError();
}

cudaError_t launch_to_bf16(const float* W, int N, int K, bf16* Wb, int ldb, cudaStream_t st) {
  k_to_bf16<<<grid_for((long long)N * ldb, 256, 152 * 32), 256, 0, st>>>(W, N, K, Wb, ldb);
  return cudaGetLastError();
}

cudaError_t launch_label_columns(const void* W, int ldw, bool w_bf16, int N, float* cols, int ldc, cudaStream_t st) {
  if (w_bf16)
    k_label_columns<bf16><<<cdiv(ldc, 256), 256, 0, st>>>((const bf16*)W, ldw, N, cols, ldc);
  else
    k_label_columns<float><<<cdiv(ldc, 256), 256, 0, st>>>((const float*)W, ldw, N, cols, ldc);
  return cudaGetLastError();
}

cudaError_t launch_expand(const float* base, int ldbase, const float* cols, const float* s1, const float* bias, int n,
                          int N, void* H, int ldh, bool h_bf16, float* s_next, float* G_acc, int* err,
                          cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  if (h_bf16)
    k_expand<bf16><<<n, 256, 0, st>>>(base, ldbase, cols, s1, bias, N, (bf16*)H, ldh, s_next, G_acc, err);
  else
    k_expand<float><<<n, 256, 0, st>>>(base, ldbase, cols, s1, bias, N, (float*)H, ldh, s_next, G_acc, err);
  return cudaGetLastError();
}

cudaError_t launch_argmax(const float* G, int n, const int* labels, int* pred, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  k_argmax<<<cdiv(n, 256), 256, 0, st>>>(G, n, labels, pred);
  return cudaGetLastError();
}

cudaError_t launch_wait_selftest(int* err, unsigned long long timeout_ns, cudaStream_t st) {
  k_wait_selftest<<<1, 32, 0, st>>>(err, timeout_ns);
  return cudaGetLastError();
}

}  // namespace ff
