// Softmax prediction head of §3 "Prediction" (Softmax method).
//
// The unlabelled input carries the neutral label (0.1 in each of the 10
// label features) and runs once through every FF layer; the activities of
// all but the first hidden layer, each normalised like a layer input
// (h / max(||h||, 1e-12)), are the features A of a linear softmax layer
// z = A V^T + c.  The head is trained by backpropagation through itself only
// (cross-entropy averaged over the rows, Adam with its own learning rate,
// §5.1): no gradient reaches the FF layers.  Prediction is the class with the
// largest logit.
//
// Kernels (all fixed-order reductions, no floating-point atomics):
//   k_head_dot     partial logits A V^T over feature splits of the
//                  segments; A is never materialised -- it is read as the
//                  stored activities H_k times their row scales s_k.  The
//                  last block of each 64-row block to finish then forms
//                  z = c + the splits' partials (in split order), softmax,
//                  per-row loss and dz = (softmax(z) - onehot(y)) / n, and
//                  the row block's partials of dc and of the loss
//   k_head_wgrad   dV partials per 64-row block: dz^T (s_k H_k)
//   k_head_adam    reduces the partials in a fixed order, Adam on V and c,
//                  the step's loss
//   k_po_grad      the Performance-Optimized step (§4): the gradient through
//                  a layer's own block into the layer and the block's dV
//                  partials; with bf16 layers it first finishes its rows'
//                  softmax from the partial logits that the forward GEMM's
//                  epilogue wrote (no k_head_dot pass)
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>

#include "ff_api_internal.h"
#include "ff_internal.cuh"
#include "ff_prof.h"
#include "ff_ptx.cuh"

namespace ff {
namespace {

constexpr int kClasses = 10;
constexpr int kMaxSegs = 16;
constexpr int kDotRows = 64;     // rows per block of k_head_dot (eight per warp)
constexpr int kSplit = 1024;     // widest feature split of one segment per k_head_dot block
constexpr int kDotMinBlocks = 152 / 2;  // k_head_dot grids narrower than this split features finer
constexpr int kWgRows = 64;      // rows per block of k_head_wgrad (8 per warp)
constexpr int kWgChunk = 128;    // features per block of k_head_wgrad (4 per lane)
constexpr int kPart = kClasses + 1;  // per-block partials: dc[10], loss

// The feature segments: segment k is layer (k+2)'s activity (layer 1's when
// there is one layer), features off[k] .. off[k] + F[k] of A, scaled per row
// by s[k] (a null s[k] reads the activity unscaled).
struct Segs {
  const void* H[kMaxSegs];
  const float* s[kMaxSegs];
  int ld[kMaxSegs];
  int F[kMaxSegs];
  int off[kMaxSegs];
  int nseg;
  int F_total;
};


// h[0..W) = H[row, f .. f+W) as float, zero past the segment or the rows.
template <typename T, int W>
__device__ __forceinline__ void load_feats(const T* __restrict__ H, int ld, int row, int n, int f, int F, float* h);
template <>
__device__ __forceinline__ void load_feats<bf16, 4>(const bf16* __restrict__ H, int ld, int row, int n, int f, int F,
                                                    float* h) {
  if (row < n && f + 4 <= F) {
    const uint2 q = __ldg(reinterpret_cast<const uint2*>(H + (size_t)row * ld + f));
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.x));
    const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.y));
    h[0] = a.x; h[1] = a.y; h[2] = b.x; h[3] = b.y;
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i)
      h[i] = (row < n && f + i < F) ? __bfloat162float(H[(size_t)row * ld + f + i]) : 0.f;
  }
}
template <>
__device__ __forceinline__ void load_feats<float, 4>(const float* __restrict__ H, int ld, int row, int n, int f, int F,
                                                     float* h) {
  if (row < n && f + 4 <= F) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(H + (size_t)row * ld + f));
    h[0] = a.x; h[1] = a.y; h[2] = a.z; h[3] = a.w;
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = (row < n && f + i < F) ? H[(size_t)row * ld + f + i] : 0.f;
  }
}

// Softmax, loss and dz of one row from its logits (z has the bias added).
// Writes logits/dz when given; returns the row's loss (0 without a label).
__device__ __forceinline__ float finish_row(const float (&z)[kClasses], int row, const int* __restrict__ labels,
                                            float inv_n, float* __restrict__ logits, float* __restrict__ dz,
                                            float (&dzr)[kClasses], int* err) {
  bool finite = true;
#pragma unroll
  for (int c = 0; c < kClasses; ++c) {
    if (logits) logits[(size_t)row * kClasses + c] = z[c];
    finite = finite && isfinite(z[c]);
    dzr[c] = 0.f;
  }
  if (!finite) atomicOr(err, DEVERR_NONFINITE);
  if (!labels) return 0.f;
  float m = z[0];
#pragma unroll
  for (int c = 1; c < kClasses; ++c) m = fmaxf(m, z[c]);
  float e[kClasses], sum = 0.f;
#pragma unroll
  for (int c = 0; c < kClasses; ++c) {
    e[c] = expf(z[c] - m);
    sum += e[c];
  }
  const int y = labels[row];
  const float inv = 1.f / sum;
  float zy = 0.f;
#pragma unroll
  for (int c = 0; c < kClasses; ++c) {
    const float p = e[c] * inv;
    dzr[c] = (p - (c == y ? 1.f : 0.f)) * inv_n;
    if (c == y) zy = z[c];
    if (dz) dz[(size_t)row * kClasses + c] = dzr[c];
  }
  return (m + logf(sum)) - zy;
}

// Number of feature splits of width `split`: segment k has ceil(F_k / split).
__host__ __device__ inline int head_splits(const int* F, int nseg, int split) {
  int S = 0;
  for (int k = 0; k < nseg; ++k) S += (F[k] + split - 1) / split;
  return S;
}

// Split width of k_head_dot for n rows: kSplit, halved (down to one 512-byte
// chunk, 512 / es features) while the grid would cover less than half the
// SMs, so that few rows are spread over the SMs by features.  (A block's
// fixed costs -- its slice of V, the cross-lane sums -- make narrower splits
// slower once the grid covers the GPU: 6000 features x 1024 rows run fastest
// at 96 blocks of 1024 features, 2000 x 1024 at 128 blocks of 256.)
int dot_split(const int* F, int nseg, int n, int es) {
  const int ch = 512 / es;
  const long long rb = (n + kDotRows - 1) / kDotRows;
  int split = kSplit;
  while (split > ch && head_splits(F, nseg, split) * rb < kDotMinBlocks) split /= 2;
  return split;
}

// Floats of partial logits k_head_dot writes for any row count up to `rows`.
size_t zpart_floats(const int* F, int nseg, int rows, int es) {
  size_t mx = 0;
  for (int rb = 1; (rb - 1) * kDotRows < rows; ++rb) {
    const int n = rb * kDotRows < rows ? rb * kDotRows : rows;
    const size_t z = (size_t)head_splits(F, nseg, dot_split(F, nseg, n, es)) * n * kClasses;
    if (z > mx) mx = z;
  }
  return mx;
}

// What the last block of a row block needs to finish its rows: the bias,
// labels (null: logits only), outputs, the head's step counter (advanced by
// row block 0 when training) and one arrival counter per row block (zero
// between launches; the finishing block resets it).
struct FinishArgs {
  const float* cb;
  const int* labels;
  float inv_n;
  float* logits;  // [n, 10] or null
  float* dz;      // [n, 10] or null
  float* part;    // [row blocks, 11] or null
  ff_dev_state* ds;
  float beta1, beta2;
  int* counter;
  int S;          // blocks (splits) per row block
};

// One tensor map per segment: H_k as [n, ld_k] with 64-row boxes of 512
// bytes (256 bf16 or 128 fp32 features), no swizzle.
struct HeadMaps {
  CUtensorMap m[kMaxSegs];
};

constexpr int kDotStages = 2;
constexpr int kDotStageBytes = kDotRows * 512;
constexpr int kDotSmem = kDotStages * kDotStageBytes + kSplit * kClasses * 4 + 64;

// zpart[split, row, c] = sum over the split's features f of s_k[row] H_k[row, f] V[c, off_k + f].
// One block per (split, 64 rows), eight rows per warp.  Thread 0 streams the
// split's 512-byte-wide row tiles of H_k into a two-stage shared-memory ring
// with TMA (mbarrier completion; a stage is refilled once all eight warps
// have arrived on its `empty` barrier); the split's slice of V sits in shared
// memory interleaved so that lane l's features (FPL consecutive ones per
// chunk) are read without bank conflicts.  Every wait is bounded.
template <typename T>
__global__ void __launch_bounds__(256, 1) k_head_dot(const __grid_constant__ HeadMaps maps, Segs sg, int split, int n,
                                                     const float* __restrict__ V, float* __restrict__ zpart,
                                                     FinishArgs fa, int* err) {
  constexpr int CH = 512 / (int)sizeof(T);  // features per chunk
  constexpr int FPL = CH / 32;              // features per lane
  constexpr int NCH = kSplit / CH;          // chunks in the widest split
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* ring = dsm;
  float* Vs = reinterpret_cast<float*>(dsm + kDotStages * kDotStageBytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(Vs + NCH * kClasses * CH);
  uint64_t* empty = full + kDotStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kDotStages);
  volatile int* never_set = abort_flag + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int k = 0, sp = blockIdx.x;
  while (k + 1 < sg.nseg && sp >= (sg.F[k] + split - 1) / split) {
    sp -= (sg.F[k] + split - 1) / split;
    ++k;
  }
  const int off = sg.off[k];
  const int fs = sp * split;
  const int fe = min(fs + split, sg.F[k]);
  const int nch = (fe - fs + CH - 1) / CH;
  const int rblk = blockIdx.y * kDotRows;
  const CUtensorMap* map = &maps.m[k];
  int issued = 0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kDotStages; ++i) {
      ptx::mbar_init(&full[i], 1);
      ptx::mbar_init(&empty[i], 8);
    }
    *abort_flag = 0;
    *never_set = 0;
    ptx::fence_mbar_init();
    ptx::prefetch_tmap(map);
  }
  __syncthreads();
  ptx::griddep_wait();  // launched with programmatic stream serialization
  if (threadIdx.x == 0) {
    for (; issued < kDotStages && issued < nch; ++issued) {
      if (!ff_dcheck(tma_x_aligned(fs + issued * CH, (int)sizeof(T)), err)) {
        *abort_flag = 1;
        break;
      }
      ptx::mbar_arrive_expect_tx(&full[issued], kDotStageBytes);
      ptx::tma_load_2d(ring + issued * kDotStageBytes, map, &full[issued], fs + issued * CH, rblk);
    }
  }
  // the split's slice of V, zero past the segment
  for (int idx = threadIdx.x; idx < nch * kClasses * CH; idx += 256) {
    const int ch = idx / (kClasses * CH), rem = idx % (kClasses * CH);
    const int c = rem / CH, j = rem % CH;
    const int f = fs + ch * CH + j;
    Vs[((ch * kClasses + c) * FPL + j % FPL) * 32 + j / FPL] = f < fe ? __ldg(V + (size_t)c * sg.F_total + off + f) : 0.f;
  }
  const int r0 = rblk + warp * 8;
  float srow[8];
#pragma unroll
  for (int r = 0; r < 8; ++r) srow[r] = (r0 + r < n) ? (sg.s[k] ? __ldg(sg.s[k] + r0 + r) : 1.f) : 0.f;
  __syncthreads();
  float acc[8][kClasses];
#pragma unroll
  for (int r = 0; r < 8; ++r)
#pragma unroll
    for (int c = 0; c < kClasses; ++c) acc[r][c] = 0.f;
  for (int ch = 0; ch < nch; ++ch) {
    const int s = ch % kDotStages;
    const uint32_t ph = (uint32_t)(ch / kDotStages) & 1u;
    if (!ptx::mbar_wait(&full[s], ph, kWaitTimeoutNs, abort_flag)) {
      *abort_flag = 1;
      atomicOr(err, DEVERR_TIMEOUT);
      break;
    }
    const uint8_t* tile = ring + s * kDotStageBytes;
    const float* vch = Vs + ch * kClasses * FPL * 32;
    // the warp's 8 rows of this chunk (scaled by s_k), then every V value
    // read once from shared memory serves all 8 rows
    float h[8][FPL];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const uint8_t* rowp = tile + (warp * 8 + r) * 512 + lane * 16;
      if constexpr (sizeof(T) == 2) {
        const uint4 q = *reinterpret_cast<const uint4*>(rowp);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
          h[r][2 * i] = v.x * srow[r];
          h[r][2 * i + 1] = v.y * srow[r];
        }
      } else {
        const float4 q = *reinterpret_cast<const float4*>(rowp);
        h[r][0] = q.x * srow[r];
        h[r][1] = q.y * srow[r];
        h[r][2] = q.z * srow[r];
        h[r][3] = q.w * srow[r];
      }
    }
#pragma unroll
    for (int c = 0; c < kClasses; ++c)
#pragma unroll
      for (int e = 0; e < FPL; ++e) {
        const float v = vch[(c * FPL + e) * 32 + lane];
#pragma unroll
        for (int r = 0; r < 8; ++r) acc[r][c] = fmaf(h[r][e], v, acc[r][c]);
      }
    __syncwarp();
    if (lane == 0) ptx::mbar_arrive(&empty[s]);
    if (threadIdx.x == 0 && issued < nch) {
      // stage s is refilled with chunk `issued` (= ch + kDotStages) once every warp is done with it
      if (!ptx::mbar_wait(&empty[s], ph, kWaitTimeoutNs, abort_flag)) {
        *abort_flag = 1;
        atomicOr(err, DEVERR_TIMEOUT);
        break;
      }
      if (!ff_dcheck(tma_x_aligned(fs + issued * CH, (int)sizeof(T)), err)) {
        *abort_flag = 1;
        break;
      }
      ptx::mbar_arrive_expect_tx(&full[s], kDotStageBytes);
      ptx::tma_load_2d(ring + s * kDotStageBytes, map, &full[s], fs + issued * CH, rblk);
      ++issued;
    }
  }
  if (*abort_flag) {
    // copies already issued land before the block's shared memory goes away
    if (threadIdx.x == 0)
      for (int ch = issued - kDotStages < 0 ? 0 : issued - kDotStages; ch < issued; ++ch)
        ptx::mbar_wait(&full[ch % kDotStages], (uint32_t)(ch / kDotStages) & 1u, 10000000ull, never_set);
  } else {
#pragma unroll
    for (int r = 0; r < 8; ++r)
#pragma unroll
      for (int c = 0; c < kClasses; ++c) acc[r][c] = warp_sum(acc[r][c]);
    // lane c writes class c of the warp's rows
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      if (lane != c) continue;
#pragma unroll
      for (int r = 0; r < 8; ++r)
        if (r0 + r < n) zpart[((size_t)blockIdx.x * n + r0 + r) * kClasses + c] = acc[r][c];
    }
  }
  // Every block arrives (an aborted one too, so that the counter is reset);
  // the last of the row block's S blocks finishes its rows.
  __shared__ int last;
  __shared__ float fred[kDotRows / 32][kPart];
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(fa.counter + blockIdx.y, 1) == fa.S - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    fa.counter[blockIdx.y] = 0;
    if (blockIdx.y == 0 && fa.labels && fa.ds) {
      // this step's Adam counter and bias corrections, read by k_head_adam
      fa.ds->t += 1;
      fa.ds->pow1 *= (double)fa.beta1;
      fa.ds->pow2 *= (double)fa.beta2;
      fa.ds->bc1 = (float)(1.0 - fa.ds->pow1);
      fa.ds->bc2 = (float)(1.0 - fa.ds->pow2);
    }
  }
  if (threadIdx.x >= kDotRows) return;
  // one thread per row: z = c + the splits' partials in split order (read
  // past L1: other blocks wrote them during this launch)
  const int row = rblk + (int)threadIdx.x;
  float dzr[kClasses];
  float loss = 0.f;
#pragma unroll
  for (int c = 0; c < kClasses; ++c) dzr[c] = 0.f;
  if (row < n) {
    float z[kClasses];
#pragma unroll
    for (int c = 0; c < kClasses; ++c) z[c] = __ldg(fa.cb + c);
    // four splits' loads in flight at a time, added in split order
    for (int sp0 = 0; sp0 < fa.S; sp0 += 4) {
      float t[4][kClasses];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float* zp = zpart + ((size_t)(sp0 + u) * n + row) * kClasses;
#pragma unroll
        for (int c = 0; c < kClasses; ++c) t[u][c] = sp0 + u < fa.S ? __ldcg(zp + c) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (sp0 + u < fa.S) {
#pragma unroll
          for (int c = 0; c < kClasses; ++c) z[c] += t[u][c];
        }
    }
    loss = finish_row(z, row, fa.labels, fa.inv_n, fa.logits, fa.dz, dzr, err);
  }
  if (!fa.part) return;
  // the row block's sums of dz (for dc) and of the loss, in a fixed order
#pragma unroll
  for (int c = 0; c < kClasses; ++c) dzr[c] = warp_sum(dzr[c]);
  loss = warp_sum(loss);
  if (lane == 0) {
#pragma unroll
    for (int c = 0; c < kClasses; ++c) fred[warp][c] = dzr[c];
    fred[warp][kClasses] = loss;
  }
  asm volatile("bar.sync 1, %0;" ::"n"(kDotRows) : "memory");  // the row block's warps only
  if (threadIdx.x < kPart) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kDotRows / 32; ++w) t += fred[w][threadIdx.x];
    fa.part[(size_t)blockIdx.y * kPart + threadIdx.x] = t;
  }
}

// dV partials of one 128-row block for one 128-feature chunk of one segment:
// dVpart[rb, c, f] = sum over the block's rows i of dz[i, c] s_k[i] H_k[i, f].
// Eight warps take 16 rows each (lane = 4 features); the eight partial sums
// are added in warp order.
template <typename T>
__global__ void __launch_bounds__(256) k_head_wgrad(Segs sg, int n, const float* __restrict__ dz,
                                                    float* __restrict__ dVpart) {
  __shared__ float dzs[kWgRows][kClasses];
  __shared__ float red[8][kClasses][kWgChunk];
  ptx::griddep_wait();  // launched with programmatic stream serialization
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // segment and chunk of this block
  int k = 0, chunk = blockIdx.x;
  while (k + 1 < sg.nseg && chunk >= (sg.F[k] + kWgChunk - 1) / kWgChunk) {
    chunk -= (sg.F[k] + kWgChunk - 1) / kWgChunk;
    ++k;
  }
  const T* H = static_cast<const T*>(sg.H[k]);
  const int ld = sg.ld[k], Fk = sg.F[k], off = sg.off[k];
  const int f0 = chunk * kWgChunk;
  const int rb0 = blockIdx.y * kWgRows;
  for (int idx = threadIdx.x; idx < kWgRows * kClasses; idx += 256) {
    const int i = idx / kClasses, c = idx % kClasses;
    const int row = rb0 + i;
    dzs[i][c] = row < n ? __ldg(dz + (size_t)row * kClasses + c) * (sg.s[k] ? __ldg(sg.s[k] + row) : 1.f) : 0.f;
  }
  __syncthreads();
  float acc[kClasses][4];
#pragma unroll
  for (int c = 0; c < kClasses; ++c)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[c][e] = 0.f;
  const int f = f0 + 4 * lane;
#pragma unroll 4
  for (int i = warp * (kWgRows / 8); i < (warp + 1) * (kWgRows / 8); ++i) {
    float h[4];
    load_feats<T, 4>(H, ld, rb0 + i, n, f, Fk, h);
#pragma unroll
    for (int c = 0; c < kClasses; ++c) {
      const float d = dzs[i][c];
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[c][e] = fmaf(d, h[e], acc[c][e]);
    }
  }
#pragma unroll
  for (int c = 0; c < kClasses; ++c)
#pragma unroll
    for (int e = 0; e < 4; ++e) red[warp][c][4 * lane + e] = acc[c][e];
  __syncthreads();
  for (int idx = threadIdx.x; idx < kClasses * kWgChunk; idx += 256) {
    const int c = idx / kWgChunk, j = idx % kWgChunk;
    if (f0 + j >= Fk) continue;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) v += red[w][c][j];
    dVpart[((size_t)blockIdx.y * kClasses + c) * sg.F_total + off + f0 + j] = v;
  }
}

// ------------------------------------------ Performance-Optimized layer (§4)
// The gradient that a layer's softmax block sends back into the layer, one
// block per 32 rows x 256 columns (block 32 x 8; thread (x, y) owns columns
// 8x..8x+7 of rows y, y+8, y+16, y+24):
//   dZ_ij = (sum_c dz_ic V_cj) [h_ij > 0],  G_ij = s_i dZ_ij (weight-gradient
//   operand, in the activity type),  db partials = sum over the block's rows,
//   and the block's own weight-gradient partials dV_cj = sum_i dz_ic h_ij
//   over the same rows (the block reads the raw activity).
// V (before this step's update) and dz are staged in shared memory.  Lead
// blocks (x == 0) also write the next layer's row scale from the forward's
// goodness partials; block (0, 0) advances the layer's Adam step.
// With zpart set (bf16 layers), dz is not given: the forward GEMM wrote the
// block's partial logits, and every block finishes its own rows from them
// (bias + partials in tile order, softmax, cross-entropy; the blocks of a row
// block compute identical values); lead blocks then write the row block's dz
// and loss sums, and block (0, 0) also advances the block's Adam step.
struct PoGradArgs {
  const float* dz;      // [n, 10], or null with zpart
  const float* zpart;   // [zt, n, 10] partial logits, or null
  int zt;
  const float* cb;      // [10] block bias
  const int* labels;    // [n]
  float inv_n;
  float* part;          // [row blocks, 11]: sums of dz and of the loss (with zpart)
  ff_dev_state* hds;    // the block's Adam state (with zpart)
  float hbeta1, hbeta2;
  const float* V;       // [10, N] (before this step's update)
  const float* s;       // [n] row scale of the layer input
  const float* gpart;   // forward goodness partials [ntiles, n]
  int ntiles, n, N, ld;
  float* s_next;        // [n] or null
  float* dbpart;        // [row blocks, N]
  float* dVpart;        // [row blocks, 10, N]: the block's dV partials
  ff_dev_state* ds;     // the layer's
  float beta1, beta2;
  int* err;
};

constexpr int kPoRows = 32;

template <typename T>
__global__ void __launch_bounds__(256) k_po_grad(PoGradArgs a, const T* __restrict__ H, T* __restrict__ G) {
  __shared__ float Vsh[kClasses][8][32];  // V[c][c0 + 8 l + e] at [c][e][l]: conflict-free reads
  __shared__ float dzs[kPoRows][kClasses];
  // the block's activity tile in its own type (for the dV partials), then
  // the db reduction in the same memory
  __shared__ __align__(16) T Hs[kPoRows][256 + 8];
  static_assert(sizeof(Hs) >= 8 * (256 + 4) * sizeof(float), "the db reduction fits in the tile's memory");
  const int r0 = blockIdx.y * kPoRows;
  const int lane = threadIdx.x, tid = threadIdx.y * 32 + threadIdx.x;
  const int c0 = blockIdx.x * 256;
  const int cg = c0 + lane * 8;
  const bool cols_ok = cg < a.ld;
  ptx::griddep_wait();  // launched with programmatic stream serialization
  // this thread's activity (rows y, y+8, y+16, y+24; 8 columns), loaded first
  // so that its latency overlaps the logits and softmax below
  float hv[4][8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int i = r0 + threadIdx.y + 8 * k;
    if (cols_ok && i < a.n) {
      Vec8<T>::load(H + (size_t)i * a.ld + cg, hv[k]);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) hv[k][e] = 0.f;
    }
  }
  for (int idx = tid; idx < kClasses * 256; idx += 256) {
    const int c = idx / 256, j = idx % 256;
    Vsh[c][j % 8][j / 8] = (c0 + j < a.N) ? __ldg(a.V + (size_t)c * a.N + c0 + j) : 0.f;
  }
  if (a.zpart) {
    // logits of the block's rows: thread per (row, class), partials in tile order
    for (int idx = tid; idx < kPoRows * kClasses; idx += 256) {
      const int i = idx / kClasses, c = idx % kClasses;
      dzs[i][c] = r0 + i < a.n ? __ldg(a.cb + c) + sum_partials(a.zpart, a.zt, a.n * kClasses, (r0 + i) * kClasses + c)
                               : 0.f;
    }
    __syncthreads();
    if (threadIdx.y == 0) {
      // warp 0: softmax, loss and dz of row r0 + lane, in place
      float z[kClasses], dzr[kClasses];
#pragma unroll
      for (int c = 0; c < kClasses; ++c) z[c] = dzs[lane][c];
      float loss = 0.f;
      if (r0 + lane < a.n) {
        loss = finish_row(z, r0 + lane, a.labels, a.inv_n, nullptr, nullptr, dzr, &a.hds->err);
      } else {
#pragma unroll
        for (int c = 0; c < kClasses; ++c) dzr[c] = 0.f;
      }
#pragma unroll
      for (int c = 0; c < kClasses; ++c) dzs[lane][c] = dzr[c];
      if (blockIdx.x == 0) {
        // the row block's sums of dz (for dc) and of the loss, in a fixed order
#pragma unroll
        for (int c = 0; c < kClasses; ++c) dzr[c] = warp_sum(dzr[c]);
        loss = warp_sum(loss);
        if (lane < kPart) {
          float t = loss;
#pragma unroll
          for (int c = 0; c < kClasses; ++c)
            if (lane == c) t = dzr[c];
          a.part[(size_t)blockIdx.y * kPart + lane] = t;
        }
        if (blockIdx.y == 0 && lane == 0) {
          a.hds->t += 1;
          a.hds->pow1 *= (double)a.hbeta1;
          a.hds->pow2 *= (double)a.hbeta2;
          a.hds->bc1 = (float)(1.0 - a.hds->pow1);
          a.hds->bc2 = (float)(1.0 - a.hds->pow2);
        }
      }
    }
  } else {
    for (int idx = tid; idx < kPoRows * kClasses; idx += 256) {
      const int i = idx / kClasses, c = idx % kClasses;
      dzs[i][c] = (r0 + i < a.n) ? __ldg(a.dz + (size_t)(r0 + i) * kClasses + c) : 0.f;
    }
  }
  if (blockIdx.x == 0 && tid < kPoRows && r0 + tid < a.n) {
    const float g = sum_partials(a.gpart, a.ntiles, a.n, r0 + tid);
    if (!isfinite(g)) atomicOr(a.err, DEVERR_NONFINITE);
    if (a.s_next) {
      const float r = sqrtf(g);
      a.s_next[r0 + tid] = r != r ? r : 1.f / fmaxf(r, 1e-12f);
    }
  }
  if (blockIdx.x == 0 && blockIdx.y == 0 && tid == 0) {
    a.ds->t += 1;
    a.ds->pow1 *= a.beta1;
    a.ds->pow2 *= a.beta2;
    a.ds->bc1 = (float)(1.0 - a.ds->pow1);
    a.ds->bc2 = (float)(1.0 - a.ds->pow2);
  }
  __syncthreads();
  float db[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) db[e] = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int li = threadIdx.y + 8 * k;
    const int i = r0 + li;
    const float(&h)[8] = hv[k];
    float z[8];
    Vec8<T>::store(&Hs[li][lane * 8], h);
    if (!cols_ok || i >= a.n) continue;
    const float si = __ldg(a.s + i);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      float d = 0.f;
#pragma unroll
      for (int c = 0; c < kClasses; ++c) d = fmaf(dzs[li][c], Vsh[c][e][lane], d);
      d = h[e] > 0.f ? d : 0.f;
      db[e] += d;
      z[e] = si * d;
    }
    Vec8<T>::store(G + (size_t)i * a.ld + cg, z);
  }
  __syncthreads();
  // dV partials from the staged tile: thread (x, y) sums classes y and
  // y + 8 (when below 10) over the block's 32 rows in order, for its 8 columns
#pragma unroll
  for (int c = threadIdx.y; c < kClasses; c += 8) {
    float dv[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) dv[e] = 0.f;
    for (int li = 0; li < kPoRows; ++li) {
      const float d = dzs[li][c];
      float h[8];
      Vec8<T>::load(&Hs[li][lane * 8], h);
#pragma unroll
      for (int e = 0; e < 8; ++e) dv[e] = fmaf(d, h[e], dv[e]);
    }
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (cg + e < a.N) a.dVpart[((size_t)blockIdx.y * kClasses + c) * a.N + cg + e] = dv[e];
  }
  __syncthreads();
  // db partials: the eight row groups added in order, through the tile's memory
  float (*red)[256 + 4] = reinterpret_cast<float (*)[256 + 4]>(&Hs[0][0]);
  Vec8<float>::store(&red[threadIdx.y][lane * 8], db);
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
  }
}

struct HeadAdamArgs {
  float *V, *mV, *vV, *c, *mc, *vc;
  const float* dVpart;  // [nrb, 10, F]
  int nrb, F;
  const float* part;    // [nlb, 11]
  int nlb;
  float inv_n;
  float lr, beta1, beta2, eps;
  const ff_dev_state* ds;
  float* loss_out;
  float* dV_out;        // [10, F] or null
  float* dc_out;        // [10] or null
};


// Threads 0 .. 10F-1 of the grid own one V element each; the last block owns
// the 10 biases (warp w: columns w and w + 8 of the partials, column 10 being
// the loss).
__global__ void __launch_bounds__(256) k_head_adam(HeadAdamArgs a) {
  ptx::griddep_wait();  // launched with programmatic stream serialization
  const float a1 = a.lr / a.ds->bc1, r2 = 1.f / a.ds->bc2;
  const int total = kClasses * a.F;
  const int vblocks = (total + 255) / 256;
  if ((int)blockIdx.x < vblocks) {
    const int idx = blockIdx.x * 256 + threadIdx.x;
    if (idx >= total) return;
    // the row blocks' partials in order, eight loads in flight
    const float g = sum_partials(a.dVpart, a.nrb, total, idx);
    if (a.dV_out) a.dV_out[idx] = g;
    float w = a.V[idx], m = a.mV[idx], v = a.vV[idx];
    adam1(w, m, v, g, a1, a.beta1, a.beta2, a.eps, r2);
    a.V[idx] = w;
    a.mV[idx] = m;
    a.vV[idx] = v;
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int col = warp; col < kPart; col += 8) {
    float t = 0.f;
    for (int b = lane; b < a.nlb; b += 32) t += __ldg(a.part + (size_t)b * kPart + col);
    t = warp_sum(t);
    if (lane != 0) continue;
    if (col == kClasses) {
      if (a.loss_out) a.loss_out[0] = t * a.inv_n;
      continue;
    }
    if (a.dc_out) a.dc_out[col] = t;
    float w = a.c[col], m = a.mc[col], v = a.vc[col];
    adam1(w, m, v, t, a1, a.beta1, a.beta2, a.eps, r2);
    a.c[col] = w;
    a.mc[col] = m;
    a.vc[col] = v;
  }
}

size_t align256(size_t b) { return (b + 255) & ~size_t(255); }

}  // namespace
}  // namespace ff

// The head object behind the opaque handle.
struct ff_head {
  ff_head_config cfg;
  int F;
  int device;
  cudaStream_t last_stream;
  float *V, *c, *mV, *vV, *mc, *vc;  // one allocation: V, mV, vV [10, F]; c, mc, vc [10]
  float *dV, *dc;                    // gradient of the last train step [10, F], [10]
  ff::ff_dev_state* ds;
  void* ws;
  size_t ws_bytes;
  int* counters;    // k_head_dot arrival counters, one per 64-row block (zero between launches)
  int counter_cap;
  // ff_head_train_epoch: a second feature workspace and a side stream, so
  // that the next pass's neutral forward runs while the head steps read the
  // current one (created on first use)
  void* ws2;
  size_t ws2_bytes;
  cudaStream_t side;
  cudaEvent_t ev_start, ev_fwd[2], ev_use[2];
  // ff_po_train_step: the block's Adam on the side stream (fork, join)
  cudaEvent_t ev_fork, ev_join;
};

namespace ff {
namespace {

// Validates the layer chain for the head and describes its feature segments
// (without buffers).  Returns FF_OK or FF_ERR_INVALID_ARG.
ff_status head_layers(const ff_head* hd, ff_layer* const* layers, int n_layers) {
  if (!layers || n_layers < 1 || n_layers > kMaxSegs + 1) return FF_ERR_INVALID_ARG;
  int F = 0;
  for (int k = 0; k < n_layers; ++k) {
    if (!layers[k]) return FF_ERR_INVALID_ARG;
    if (layers[k]->is_bf16 != layers[0]->is_bf16) return FF_ERR_INVALID_ARG;
    if (k > 0 && layers[k]->K != layers[k - 1]->N) return FF_ERR_INVALID_ARG;
    if (k >= 1 || n_layers == 1) F += layers[k]->N;
  }
  if (layers[0]->K < kClasses) return FF_ERR_INVALID_ARG;
  if (F != hd->F) return FF_ERR_INVALID_ARG;
  return FF_OK;
}

struct HeadWork {
  void* X0;
  float* S[kMaxSegs + 2];   // S[k]: row scale of layer k's input (S[L]: of the last activity)
  void* Hk[kMaxSegs + 1];
  float* gpart;
  float* gpart2;   // the tensor-core forward alternates between gpart and gpart2
  float* logits;
  float* zpart;
  float* dz;
  float* part;
  float* dVpart;
};

// Partial-logit floats for up to `rows` rows of the layer chain's segments.
size_t chain_zpart_floats(ff_layer* const* layers, int L, int rows) {
  int F[kMaxSegs + 1], nseg = 0;
  for (int k = (L == 1 ? 0 : 1); k < L; ++k) F[nseg++] = layers[k]->N;
  return zpart_floats(F, nseg, rows, layers[0]->is_bf16 ? 2 : 4);
}

// Carves the head's workspace for `rows` rows (grown on demand); buf 1: the
// second workspace of ff_head_train_epoch.
ff_status head_workspace(ff_head* hd, ff_layer* const* layers, int L, int rows, bool train, HeadWork* w,
                         int buf = 0) {
  void*& wsp = buf ? hd->ws2 : hd->ws;
  size_t& wsb = buf ? hd->ws2_bytes : hd->ws_bytes;
  const bool b16 = layers[0]->is_bf16;
  const size_t es = b16 ? 2 : 4;
  int ntmax = 0;
  for (int k = 0; k < L; ++k) {
    const int nt = b16 ? tc_fwd_ntiles_max(layers[k]->N) : simt_fwd_ntiles(layers[k]->N);
    if (nt > ntmax) ntmax = nt;
  }
  size_t off = 0;
  size_t oX = off; off += align256((size_t)rows * layers[0]->ldK * es);
  size_t oS[kMaxSegs + 2];
  for (int k = 0; k <= L; ++k) { oS[k] = off; off += align256((size_t)rows * 4); }
  size_t oH[kMaxSegs + 1];
  for (int k = 0; k < L; ++k) { oH[k] = off; off += align256((size_t)rows * layers[k]->ldN * es); }
  size_t oG = off; off += align256((size_t)ntmax * rows * 4);
  size_t oG2 = off; off += align256(b16 ? (size_t)ntmax * rows * 4 : 0);
  size_t oZ = off; off += align256((size_t)rows * kClasses * 4);
  size_t oZP = off; off += align256(chain_zpart_floats(layers, L, rows) * 4);
  size_t oD = off; off += align256(train ? (size_t)rows * kClasses * 4 : 0);
  size_t oP = off; off += align256(train ? (size_t)cdiv(rows, kDotRows) * kPart * 4 : 0);
  size_t oV = off; off += align256(train ? (size_t)cdiv(rows, kWgRows) * kClasses * hd->F * 4 : 0);
  if (off > wsb) {
    FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync before head workspace growth");
    if (hd->side) FF_TRY(cudaStreamSynchronize(hd->side), "sync before head workspace growth");
    dev_free(wsp);
    wsp = nullptr;
    wsb = 0;
    FF_TRY(dev_alloc(&wsp, off), "head workspace");
    wsb = off;
  }
  char* base = static_cast<char*>(wsp);
  w->X0 = base + oX;
  for (int k = 0; k <= L; ++k) w->S[k] = reinterpret_cast<float*>(base + oS[k]);
  for (int k = 0; k < L; ++k) w->Hk[k] = base + oH[k];
  w->gpart = reinterpret_cast<float*>(base + oG);
  w->gpart2 = reinterpret_cast<float*>(base + (b16 ? oG2 : oG));
  w->logits = reinterpret_cast<float*>(base + oZ);
  w->zpart = reinterpret_cast<float*>(base + oZP);
  w->dz = train ? reinterpret_cast<float*>(base + oD) : nullptr;
  w->part = train ? reinterpret_cast<float*>(base + oP) : nullptr;
  w->dVpart = train ? reinterpret_cast<float*>(base + oV) : nullptr;
  return FF_OK;
}

// Neutral-labelled forward of `rows` raw input rows through every layer:
// H_k and the row scale of every activity.  narrow: the forward GEMMs may take
// 128-column tiles when their grid is small (predict); training keeps
// 256-column tiles at every row count, so that a row's goodness partials --
// and with them every activity scale -- do not depend on how many rows share
// the GEMM (ff_head_train_epoch runs many steps' rows at once).
ff_status head_forward(ff_layer* const* layers, int L, const float* x, int rows, const HeadWork& w, int* err,
                       cudaStream_t st, bool narrow) {
  ff_layer* L0 = layers[0];
  const bool b16 = L0->is_bf16;
  const double es = b16 ? 2.0 : 4.0;
  FF_LAUNCH(K_OVERLAY, (double)rows * (L0->K * 4.0 + L0->ldK * es + 4), st,
            launch_overlay(x, nullptr, rows, L0->K, w.X0, L0->ldK, b16, w.S[0], 2, st), "neutral-label overlay");
  const void* in = w.X0;
  int nt_prev = 0;
  for (int k = 0; k < L; ++k) {
    ff_layer* Lk = layers[k];
    float* gpart = b16 && (k & 1) ? w.gpart2 : w.gpart;
    EpiArgs ep{w.S[k], Lk->cfg.has_bias ? Lk->b : nullptr, w.Hk[k], Lk->ldN, gpart};
    ep.narrow = narrow;
    int nt;
    if (b16) {
      if (k >= 1) {
        // layer k-1's activity scale S[k] comes from its goodness partials
        // inside this GEMM (no separate finalize)
        ep.row_scale = nullptr;
        ep.gpart_in = (k - 1) & 1 ? w.gpart2 : w.gpart;
        ep.ntiles_in = nt_prev;
        ep.s_out = w.S[k];
      }
      nt = tc_fwd_ntiles(rows, Lk->N, narrow);
      FF_LAUNCH(K_FWD_TC, 2.0 * rows * Lk->N * Lk->K, st,
                tc_gemm_fwd(static_cast<const bf16*>(in), Lk->ldK, Lk->Wb, Lk->ldK, rows, Lk->N, Lk->K, ep, err, st),
                "head forward GEMM (tcgen05)");
    } else {
      nt = simt_fwd_ntiles(Lk->N);
      FF_LAUNCH(K_FWD_SIMT, 2.0 * rows * Lk->N * Lk->K, st,
                simt_gemm_fwd(static_cast<const float*>(in), Lk->ldK, Lk->W, Lk->K, rows, Lk->N, Lk->K, ep, st),
                "head forward GEMM (fp32)");
    }
    nt_prev = nt;
    if (!b16 || k + 1 == L) {
      FinalizeArgs fa{};
      fa.gpart = gpart;
      fa.ntiles = nt;
      fa.M = rows;
      fa.s_next = w.S[k + 1];
      fa.err = err;
      FF_LAUNCH(K_FINALIZE, (double)rows * (nt * 4.0 + 4), st, launch_finalize(fa, st), "head activity scale");
    }
    in = w.Hk[k];
  }
  return FF_OK;
}

Segs make_segs(ff_layer* const* layers, int L, const HeadWork& w, int F) {
  Segs sg{};
  int off = 0, j = 0;
  for (int k = (L == 1 ? 0 : 1); k < L; ++k, ++j) {
    sg.H[j] = w.Hk[k];
    sg.s[j] = w.S[k + 1];
    sg.ld[j] = layers[k]->ldN;
    sg.F[j] = layers[k]->N;
    sg.off[j] = off;
    off += layers[k]->N;
  }
  sg.nseg = j;
  sg.F_total = F;
  return sg;
}

// One arrival counter per 64-row block of k_head_dot, all zero (grown on
// demand; the kernel leaves them zero).
ff_status ensure_counters(ff_head* hd, int blocks) {
  if (blocks <= hd->counter_cap) return FF_OK;
  FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync before counter growth");
  dev_free(hd->counters);
  hd->counters = nullptr;
  hd->counter_cap = 0;
  FF_TRY(dev_alloc(reinterpret_cast<void**>(&hd->counters), (size_t)blocks * sizeof(int)), "head counters");
  FF_TRY(cudaMemset(hd->counters, 0, (size_t)blocks * sizeof(int)), "zero head counters");
  hd->counter_cap = blocks;
  return FF_OK;
}

// Logits (and, with labels, softmax, loss, dz and the per-row-block
// partials) of n rows: k_head_dot over the feature splits, whose last block
// per row block finishes the rows.
ff_status head_logits(ff_head* hd, const Segs& sg, bool b16, int n, const int* labels, float* logits, float* zpart,
                      float* dz, float* part, int* err, cudaStream_t st) {
  const int es = b16 ? 2 : 4;
  const int split = dot_split(sg.F, sg.nseg, n, es);
  const int S = head_splits(sg.F, sg.nseg, split);
  ff_status s = ensure_counters(hd, cdiv(n, kDotRows));
  if (s != FF_OK) return s;
  FinishArgs fa{};
  fa.cb = hd->c;
  fa.labels = labels;
  fa.inv_n = 1.f / (float)n;
  fa.logits = logits;
  fa.dz = dz;
  fa.part = part;
  fa.ds = labels ? hd->ds : nullptr;
  fa.beta1 = hd->cfg.beta1;
  fa.beta2 = hd->cfg.beta2;
  fa.counter = hd->counters;
  fa.S = S;
  const float* V = hd->V;
  HeadMaps maps;
  std::memset(&maps, 0, sizeof(maps));
  for (int k = 0; k < sg.nseg; ++k)
    if (!make_plain_map(&maps.m[k], sg.H[k], es, sg.ld[k], n, sg.ld[k], 512 / es, kDotRows))
      return FF_ERR_INVALID_ARG;
  static const cudaError_t attr_b = cudaFuncSetAttribute(k_head_dot<bf16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                         kDotSmem);
  static const cudaError_t attr_f = cudaFuncSetAttribute(k_head_dot<float>,
                                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kDotSmem);
  FF_TRY(b16 ? attr_b : attr_f, "head kernel attributes");
  dim3 grid(S, cdiv(n, kDotRows));
  PdlLaunch l(grid, dim3(256), st, kDotSmem);
  FF_LAUNCH(K_HEAD_LOGITS, (double)n * sg.F_total * es + (double)n * (2 * S + 2) * kClasses * 4, st,
            (b16 ? cudaLaunchKernelEx(&l.cfg, k_head_dot<bf16>, maps, sg, split, n, V, zpart, fa, err)
                 : cudaLaunchKernelEx(&l.cfg, k_head_dot<float>, maps, sg, split, n, V, zpart, fa, err)),
            "head logits, softmax and cross-entropy");
  return FF_OK;
}

cudaError_t launch_head_wgrad(const Segs& sg, bool b16, int n, const float* dz, float* dVpart, cudaStream_t st) {
  int chunks = 0;
  for (int k = 0; k < sg.nseg; ++k) chunks += cdiv(sg.F[k], kWgChunk);
  PdlLaunch l(dim3(chunks, cdiv(n, kWgRows)), dim3(256), st);
  return b16 ? cudaLaunchKernelEx(&l.cfg, k_head_wgrad<bf16>, sg, n, dz, dVpart)
             : cudaLaunchKernelEx(&l.cfg, k_head_wgrad<float>, sg, n, dz, dVpart);
}

}  // namespace
}  // namespace ff

using namespace ff;

namespace ff {

int head_features(const ff_head* h) { return h->F; }
void head_forget_stream(ff_head* h, cudaStream_t st) {
  if (h->last_stream == st) h->last_stream = nullptr;
}

namespace {

// Scratch of a softmax block for n rows of a layer of width N, carved from
// the head's workspace (grown on demand).
struct PoWork {
  float *zpart, *dz, *part, *dVpart;
};

ff_status po_workspace(ff_head* hd, int n, int N, int es, PoWork* w) {
  size_t off = 0;
  // partial logits: k_head_dot's (fp32 layers) or the forward GEMM's (bf16)
  size_t zf = zpart_floats(&N, 1, n, es);
  if (es == 2) zf = std::max(zf, (size_t)tc_fwd_ntiles_max(N) * n * kClasses);
  const size_t oZ = off; off += align256(zf * 4);
  const size_t oD = off; off += align256((size_t)n * kClasses * 4);
  const size_t oP = off; off += align256((size_t)cdiv(n, std::min(kDotRows, kPoRows)) * kPart * 4);
  const size_t oV = off; off += align256((size_t)cdiv(n, kPoRows) * kClasses * N * 4);
  if (off > hd->ws_bytes) {
    FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync before workspace growth");
    if (hd->side) FF_TRY(cudaStreamSynchronize(hd->side), "sync before workspace growth");
    dev_free(hd->ws);
    hd->ws = nullptr;
    hd->ws_bytes = 0;
    FF_TRY(dev_alloc(&hd->ws, off), "block workspace");
    hd->ws_bytes = off;
  }
  char* base = static_cast<char*>(hd->ws);
  w->zpart = reinterpret_cast<float*>(base + oZ);
  w->dz = reinterpret_cast<float*>(base + oD);
  w->part = reinterpret_cast<float*>(base + oP);
  w->dVpart = reinterpret_cast<float*>(base + oV);
  return FF_OK;
}

// Adam arguments of the head / block from its state and this step's partials.
HeadAdamArgs head_adam_args(ff_head* hd, const float* dVpart, int nrb, const float* part, int nlb, int n,
                            float* loss) {
  HeadAdamArgs a{};
  a.V = hd->V;
  a.mV = hd->mV;
  a.vV = hd->vV;
  a.c = hd->c;
  a.mc = hd->mc;
  a.vc = hd->vc;
  a.dVpart = dVpart;
  a.nrb = nrb;
  a.F = hd->F;
  a.part = part;
  a.nlb = nlb;
  a.inv_n = 1.f / (float)n;
  a.lr = hd->cfg.lr;
  a.beta1 = hd->cfg.beta1;
  a.beta2 = hd->cfg.beta2;
  a.eps = hd->cfg.eps;
  a.ds = hd->ds;
  a.loss_out = loss ? loss : &hd->ds->loss;
  a.dV_out = hd->dV;
  a.dc_out = hd->dc;
  return a;
}

}  // namespace
}  // namespace ff

extern "C" {

ff_status ff_head_create(const ff_head_config* cfg, ff_head** out) {
  if (!out) return FF_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || cfg->n_features < 1 || cfg->max_rows < 0) return FF_ERR_INVALID_ARG;
  if (!std::isfinite(cfg->lr) || !(cfg->beta1 >= 0.f && cfg->beta1 < 1.f) || !(cfg->beta2 >= 0.f && cfg->beta2 < 1.f) ||
      !(cfg->eps > 0.f))
    return FF_ERR_INVALID_ARG;
  ff_head* hd = new (std::nothrow) ff_head();
  if (!hd) return FF_ERR_OOM;
  hd->cfg = *cfg;
  if (hd->cfg.max_rows == 0) hd->cfg.max_rows = 4096;
  hd->F = cfg->n_features;
  cudaGetDevice(&hd->device);
  const size_t nv = (size_t)kClasses * hd->F;
  const size_t total = 4 * nv + 5 * kClasses;  // V, mV, vV, dV; c, mc, vc, dc (+ pad)
  void* p = nullptr;
  ff_status s = cuda_status(dev_alloc(&p, total * 4), "head parameters");
  if (s != FF_OK) {
    delete hd;
    return s;
  }
  float* f = static_cast<float*>(p);
  hd->V = f;
  hd->mV = f + nv;
  hd->vV = f + 2 * nv;
  hd->dV = f + 3 * nv;
  hd->c = f + 4 * nv;
  hd->mc = hd->c + kClasses;
  hd->vc = hd->mc + kClasses;
  hd->dc = hd->vc + kClasses;
  void* dsp = nullptr;
  s = cuda_status(dev_alloc(&dsp, sizeof(ff_dev_state)), "head device state");
  if (s != FF_OK) {
    dev_free(p);
    delete hd;
    return s;
  }
  hd->ds = static_cast<ff_dev_state*>(dsp);
  const ff_dev_state init{0, 1.0, 1.0, 0.f, 0.f, 0, 0.f};
  cudaError_t e = cudaMemcpy(hd->ds, &init, sizeof(init), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(p, 0, total * 4);  // V and c start at zero (the head's reading)
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    dev_free(p);
    dev_free(dsp);
    delete hd;
    return cuda_status(e, "head initialisation");
  }
  *out = hd;
  return FF_OK;
}

ff_status ff_head_destroy(ff_head* hd) {
  if (!hd) return FF_OK;
  cudaStreamSynchronize(hd->last_stream);
  if (hd->side) {
    cudaStreamSynchronize(hd->side);
    cudaStreamDestroy(hd->side);
    cudaEventDestroy(hd->ev_start);
    cudaEventDestroy(hd->ev_fork);
    cudaEventDestroy(hd->ev_join);
    for (int i = 0; i < 2; ++i) {
      cudaEventDestroy(hd->ev_fwd[i]);
      cudaEventDestroy(hd->ev_use[i]);
    }
  }
  dev_free(hd->ws2);
  dev_free(hd->ws);
  dev_free(hd->counters);
  dev_free(hd->V);
  dev_free(hd->ds);
  delete hd;
  return FF_OK;
}

// Rows of stored features ff_head_train_epoch forms per forward pass.
constexpr int kEpochFeatureRows = 16384;

// The head's side stream and its events (created on first use).
static ff_status ensure_side(ff_head* hd) {
  if (hd->side) return FF_OK;
  FF_TRY(cudaStreamCreateWithFlags(&hd->side, cudaStreamNonBlocking), "head side stream");
  cudaEvent_t* evs[] = {&hd->ev_start, &hd->ev_fork, &hd->ev_join, &hd->ev_fwd[0], &hd->ev_fwd[1], &hd->ev_use[0],
                        &hd->ev_use[1]};
  for (cudaEvent_t* e : evs) FF_TRY(cudaEventCreateWithFlags(e, cudaEventDisableTiming), "head event");
  return FF_OK;
}

// The head's part of one train step on n rows of the features in w, starting
// at row r0 of the stored activities: logits, softmax, loss and dz
// (k_head_dot), dV partials (k_head_wgrad), Adam on V and c (k_head_adam).
static ff_status head_step_on_features(ff_head* hd, ff_layer* const* layers, int n_layers, const HeadWork& w, int r0,
                                       const int* labels, int n, float* loss, cudaStream_t st) {
  Segs sg = make_segs(layers, n_layers, w, hd->F);
  const bool b16 = layers[0]->is_bf16;
  const double es = b16 ? 2.0 : 4.0;
  for (int j = 0; j < sg.nseg; ++j) {
    sg.H[j] = static_cast<const char*>(sg.H[j]) + (size_t)r0 * sg.ld[j] * (size_t)es;
    sg.s[j] += r0;
  }
  int* err = &hd->ds->err;
  ff_status s = head_logits(hd, sg, b16, n, labels, nullptr, w.zpart, w.dz, w.part, err, st);
  if (s != FF_OK) return s;
  FF_LAUNCH(K_HEAD_WGRAD, (double)n * hd->F * es + (double)cdiv(n, kWgRows) * kClasses * hd->F * 4, st,
            launch_head_wgrad(sg, b16, n, w.dz, w.dVpart, st), "head weight gradient");
  const HeadAdamArgs a = head_adam_args(hd, w.dVpart, cdiv(n, kWgRows), w.part, cdiv(n, kDotRows), n, loss);
  const int vblocks = cdiv((long long)kClasses * hd->F, 256);
  PdlLaunch l(dim3(vblocks + 1), dim3(256), st);
  FF_LAUNCH(K_HEAD_ADAM, (double)kClasses * hd->F * (a.nrb * 4.0 + 28), st, cudaLaunchKernelEx(&l.cfg, k_head_adam, a),
            "head Adam");
  return FF_OK;
}

ff_status ff_head_train_step(ff_head* hd, ff_layer* const* layers, int n_layers, const float* x, const int* labels,
                             int n, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_head_train_step");
  if (!hd || n < 0) return FF_ERR_INVALID_ARG;
  ff_status s = head_layers(hd, layers, n_layers);
  if (s != FF_OK) return s;
  if (n == 0) return FF_OK;
  if (!x || !labels || n > hd->cfg.max_rows) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  HeadWork w;
  s = head_workspace(hd, layers, n_layers, n, true, &w);
  if (s != FF_OK) return s;
  hd->last_stream = st;
  int* err = &hd->ds->err;
  s = head_forward(layers, n_layers, x, n, w, err, st, false);
  if (s != FF_OK) return s;
  return head_step_on_features(hd, layers, n_layers, w, 0, labels, n, loss, st);
}

ff_status ff_head_train_epoch(ff_head* hd, ff_layer* const* layers, int n_layers, const float* x, const int* labels,
                              int n, int B, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_head_train_epoch");
  if (!hd || n < 0 || B < 1) return FF_ERR_INVALID_ARG;
  ff_status s = head_layers(hd, layers, n_layers);
  if (s != FF_OK) return s;
  if (n == 0) return FF_OK;
  if (!x || !labels || B > hd->cfg.max_rows) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // Rows whose features one forward pass forms: whole steps, up to
  // kEpochFeatureRows (at least one step).
  const int steps_per_chunk = kEpochFeatureRows / B > 0 ? kEpochFeatureRows / B : 1;
  const int R = (int)((long long)steps_per_chunk * B < n ? (long long)steps_per_chunk * B : n);
  const int npass = cdiv(n, R);
  if (npass > 1) {
    s = ensure_side(hd);
    if (s != FF_OK) return s;
  }
  HeadWork w[2];
  for (int i = 0; i < (npass > 1 ? 2 : 1); ++i) {
    s = head_workspace(hd, layers, n_layers, R, true, &w[i], i);
    if (s != FF_OK) return s;
  }
  hd->last_stream = st;
  int* err = &hd->ds->err;
  const int K0 = layers[0]->K;
  // Pass p's forward fills workspace p % 2 on the side stream (after the
  // head steps of pass p - 2 have read it); its head steps run on `stream`
  // after that forward, while the side stream forms pass p + 1.  One pass:
  // everything on `stream`.
  cudaStream_t fs = npass > 1 ? hd->side : st;
  if (npass > 1) {
    FF_TRY(cudaEventRecord(hd->ev_start, st), "event record");
    FF_TRY(cudaStreamWaitEvent(fs, hd->ev_start, 0), "stream wait");
  }
  for (int p = 0, r0 = 0, t = 0; p < npass; ++p, r0 += R) {
    const int rows = n - r0 < R ? n - r0 : R;
    const int buf = p & 1;
    if (npass > 1 && p >= 2) FF_TRY(cudaStreamWaitEvent(fs, hd->ev_use[buf], 0), "stream wait");
    s = head_forward(layers, n_layers, x + (size_t)r0 * K0, rows, w[buf], err, fs, false);
    if (s != FF_OK) return s;
    if (npass > 1) {
      FF_TRY(cudaEventRecord(hd->ev_fwd[buf], fs), "event record");
      FF_TRY(cudaStreamWaitEvent(st, hd->ev_fwd[buf], 0), "stream wait");
    }
    for (int q = 0; q < rows; q += B, ++t) {
      const int b = rows - q < B ? rows - q : B;
      s = head_step_on_features(hd, layers, n_layers, w[buf], q, labels + r0 + q, b, loss ? loss + t : nullptr, st);
      if (s != FF_OK) return s;
    }
    if (npass > 1) FF_TRY(cudaEventRecord(hd->ev_use[buf], st), "event record");
  }
  return FF_OK;
}

ff_status ff_head_predict(ff_head* hd, ff_layer* const* layers, int n_layers, const float* x, int n, int* pred,
                          float* logits, void* stream) {
  ff::NvtxRange nvtx_("ff_head_predict");
  if (!hd || n < 0) return FF_ERR_INVALID_ARG;
  ff_status s = head_layers(hd, layers, n_layers);
  if (s != FF_OK) return s;
  if (n == 0) return FF_OK;
  if (!x || (!pred && !logits)) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int C = n < hd->cfg.max_rows ? n : hd->cfg.max_rows;
  HeadWork w;
  s = head_workspace(hd, layers, n_layers, C, false, &w);
  if (s != FF_OK) return s;
  hd->last_stream = st;
  int* err = &hd->ds->err;
  const bool b16 = layers[0]->is_bf16;
  const int K0 = layers[0]->K;
  for (int r0 = 0; r0 < n; r0 += C) {
    const int cn = (n - r0) < C ? (n - r0) : C;
    s = head_forward(layers, n_layers, x + (size_t)r0 * K0, cn, w, err, st, true);
    if (s != FF_OK) return s;
    const Segs sg = make_segs(layers, n_layers, w, hd->F);
    float* z = logits ? logits + (size_t)r0 * kClasses : w.logits;
    s = head_logits(hd, sg, b16, cn, nullptr, z, w.zpart, nullptr, nullptr, err, st);
    if (s != FF_OK) return s;
    if (pred)
      FF_LAUNCH(K_ARGMAX, (double)cn * 44, st, launch_argmax(z, cn, nullptr, pred + r0, st), "head argmax");
  }
  return FF_OK;
}

static ff_status head_copy(void* dst, const void* src, size_t bytes) {
  if (!dst || !src) return FF_OK;
  FF_TRY(cudaMemcpy(dst, src, bytes, cudaMemcpyDefault), "head state copy");
  return FF_OK;
}

ff_status ff_head_get_state(const ff_head* hdc, float* V, float* c, float* mV, float* vV, float* mc, float* vc,
                            long long* step) {
  if (!hdc) return FF_ERR_INVALID_ARG;
  ff_head* hd = const_cast<ff_head*>(hdc);
  FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync");
  const size_t nv = (size_t)kClasses * hd->F * 4, nc = kClasses * 4;
  ff_status s;
  if ((s = head_copy(V, hd->V, nv)) != FF_OK) return s;
  if ((s = head_copy(mV, hd->mV, nv)) != FF_OK) return s;
  if ((s = head_copy(vV, hd->vV, nv)) != FF_OK) return s;
  if ((s = head_copy(c, hd->c, nc)) != FF_OK) return s;
  if ((s = head_copy(mc, hd->mc, nc)) != FF_OK) return s;
  if ((s = head_copy(vc, hd->vc, nc)) != FF_OK) return s;
  if (step) {
    ff_dev_state d;
    FF_TRY(cudaMemcpy(&d, hd->ds, sizeof(d), cudaMemcpyDeviceToHost), "head step counter");
    *step = d.t;
  }
  return FF_OK;
}

ff_status ff_head_set_state(ff_head* hd, const float* V, const float* c, const float* mV, const float* vV,
                            const float* mc, const float* vc, long long step) {
  if (!hd || step < 0) return FF_ERR_INVALID_ARG;
  FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync");
  const size_t nv = (size_t)kClasses * hd->F * 4, nc = kClasses * 4;
  ff_status s;
  if ((s = head_copy(hd->V, V, nv)) != FF_OK) return s;
  if ((s = head_copy(hd->mV, mV, nv)) != FF_OK) return s;
  if ((s = head_copy(hd->vV, vV, nv)) != FF_OK) return s;
  if ((s = head_copy(hd->c, c, nc)) != FF_OK) return s;
  if ((s = head_copy(hd->mc, mc, nc)) != FF_OK) return s;
  if ((s = head_copy(hd->vc, vc, nc)) != FF_OK) return s;
  ff_dev_state d;
  FF_TRY(cudaMemcpy(&d, hd->ds, sizeof(d), cudaMemcpyDeviceToHost), "head device state");
  d.t = step;
  d.pow1 = std::pow((double)hd->cfg.beta1, (double)step);
  d.pow2 = std::pow((double)hd->cfg.beta2, (double)step);
  FF_TRY(cudaMemcpy(hd->ds, &d, sizeof(d), cudaMemcpyHostToDevice), "head device state");
  return FF_OK;
}

ff_status ff_head_get_grad(const ff_head* hdc, float* dV, float* dc) {
  if (!hdc) return FF_ERR_INVALID_ARG;
  ff_head* hd = const_cast<ff_head*>(hdc);
  FF_TRY(cudaStreamSynchronize(hd->last_stream), "sync");
  ff_status s;
  if ((s = head_copy(dV, hd->dV, (size_t)kClasses * hd->F * 4)) != FF_OK) return s;
  return head_copy(dc, hd->dc, kClasses * 4);
}

ff_status ff_head_check(ff_head* hd) {
  if (!hd) return FF_ERR_INVALID_ARG;
  FF_TRY(cudaStreamSynchronize(hd->last_stream), "check sync");
  int err = 0;
  FF_TRY(cudaMemcpy(&err, &hd->ds->err, sizeof(int), cudaMemcpyDeviceToHost), "read error word");
  if (err) {
    const int zero = 0;
    FF_TRY(cudaMemcpy(&hd->ds->err, &zero, sizeof(int), cudaMemcpyHostToDevice), "clear error word");
  }
  if (err & DEVERR_CHECK) return FF_ERR_DEVICE_CHECK;  // a skipped copy also runs waits out
  if (err & DEVERR_TIMEOUT) return FF_ERR_TIMEOUT;
  if (err & DEVERR_NONFINITE) return FF_ERR_NONFINITE;
  return FF_OK;
}

// ------------------------------------------ Performance-Optimized layer (§4)
ff_status ff_po_train_step(ff_layer* L, ff_head* hd, const void* x, int raw_input, const float* row_scale,
                           const int* labels, int n, void* h_out, float* next_scale, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_po_train_step");
  if (!L || !hd || n < 0) return FF_ERR_INVALID_ARG;
  if (hd->F != L->N) return FF_ERR_INVALID_ARG;
  if (raw_input && L->K < kClasses) return FF_ERR_INVALID_ARG;
  if (n == 0) return FF_OK;
  if (!x || !labels) return FF_ERR_INVALID_ARG;
  if (h_out && (reinterpret_cast<uintptr_t>(h_out) & 15u)) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ff_status s = ensure_capacity(L, n);
  if (s != FF_OK) return s;
  PoWork w;
  s = po_workspace(hd, n, L->N, L->is_bf16 ? 2 : 4, &w);
  if (s != FF_OK) return s;
  L->last_stream = st;
  hd->last_stream = st;
  const bool b16 = L->is_bf16;
  const double es = b16 ? 2.0 : 4.0;
  const int K = L->K, N = L->N;
  // the layer's forward pass (layer 1: the neutral-labelled raw input)
  const void* X;
  const float* sc;
  if (raw_input) {
    FF_LAUNCH(K_OVERLAY, (double)n * (K * 4.0 + L->ldK * es + 4), st,
              launch_overlay(static_cast<const float*>(x), nullptr, n, K, L->X, L->ldK, b16, L->s_in, 2, st),
              "neutral-label overlay");
    X = L->X;
    sc = L->s_in;
  } else {
    X = x;
    if (row_scale) {
      sc = row_scale;
    } else {
      FF_LAUNCH(K_ROW_SCALE, (double)n * (K * es + 4), st, launch_row_scale(x, L->ldK, b16, n, K, L->s_in, st),
                "row scale");
      sc = L->s_in;
    }
  }
  void* H = h_out ? h_out : L->H;
  EpiArgs ep{sc, L->cfg.has_bias ? L->b : nullptr, H, L->ldN, L->gpart};
  int ntiles;
  if (b16) {
    // the block's partial logits come out of the forward GEMM's epilogue
    ep.logit_V = hd->V;
    ep.logit_ldV = N;
    ep.zpart = w.zpart;
    ntiles = tc_fwd_ntiles(n, N, false);
    FF_LAUNCH(K_FWD_TC, 2.0 * n * N * K, st,
              tc_gemm_fwd(static_cast<const bf16*>(X), L->ldK, L->Wb, L->ldK, n, N, K, ep, &L->ds->err, st),
              "forward GEMM (tcgen05)");
  } else {
    ntiles = simt_fwd_ntiles(N);
    FF_LAUNCH(K_FWD_SIMT, 2.0 * n * N * K, st,
              simt_gemm_fwd(static_cast<const float*>(X), L->ldK, L->W, K, n, N, K, ep, st), "forward GEMM (fp32)");
  }
  if (!b16) {
    // the block on the raw activity: logits, cross-entropy, dz
    Segs sg{};
    sg.H[0] = H;
    sg.s[0] = nullptr;
    sg.ld[0] = L->ldN;
    sg.F[0] = N;
    sg.off[0] = 0;
    sg.nseg = 1;
    sg.F_total = N;
    s = head_logits(hd, sg, b16, n, labels, nullptr, w.zpart, w.dz, w.part, &hd->ds->err, st);
    if (s != FF_OK) return s;
  }
  // the gradient reaching the layer, with the block's weights before its
  // update, and the block's weight-gradient partials (bf16: after finishing
  // the block's rows from the GEMM's partial logits)
  PoGradArgs pa{};
  if (b16) {
    pa.zpart = w.zpart;
    pa.zt = ntiles;
    pa.cb = hd->c;
    pa.labels = labels;
    pa.inv_n = 1.f / (float)n;
    pa.part = w.part;
    pa.hds = hd->ds;
    pa.hbeta1 = hd->cfg.beta1;
    pa.hbeta2 = hd->cfg.beta2;
  } else {
    pa.dz = w.dz;
  }
  pa.V = hd->V;
  pa.s = sc;
  pa.gpart = L->gpart;
  pa.ntiles = ntiles;
  pa.n = n;
  pa.N = N;
  pa.ld = L->ldN;
  pa.s_next = next_scale;
  pa.dbpart = L->dbpart;
  pa.dVpart = w.dVpart;
  pa.ds = L->ds;
  pa.beta1 = L->cfg.beta1;
  pa.beta2 = L->cfg.beta2;
  pa.err = &L->ds->err;
  PdlLaunch pl(dim3(cdiv(L->ldN, 256), cdiv(n, kPoRows)), dim3(32, 8), st);
  FF_LAUNCH(K_GRAD_PREP, (double)n * L->ldN * es * 2 + (double)cdiv(n, kPoRows) * (kClasses + 1) * N * 4, st,
            (b16 ? cudaLaunchKernelEx(&pl.cfg, k_po_grad<bf16>, pa, static_cast<const bf16*>(H),
                                      static_cast<bf16*>(L->dZ))
                 : cudaLaunchKernelEx(&pl.cfg, k_po_grad<float>, pa, static_cast<const float*>(H),
                                      static_cast<float*>(L->dZ))),
            "block gradient into the layer");
  // The block's Adam needs only what k_po_grad wrote, and nothing later in
  // this step reads the block's weights: it runs on the head's side stream,
  // beside the layer's weight gradient and Adam, and `stream` joins it at the
  // end of the step.
  s = ensure_side(hd);
  if (s != FF_OK) return s;
  FF_TRY(cudaEventRecord(hd->ev_fork, st), "event record");
  FF_TRY(cudaStreamWaitEvent(hd->side, hd->ev_fork, 0), "stream wait");
  {
    const HeadAdamArgs ha =
        head_adam_args(hd, w.dVpart, cdiv(n, kPoRows), w.part, cdiv(n, b16 ? kPoRows : kDotRows), n, loss);
    const int vblocks = cdiv((long long)kClasses * hd->F, 256);
    // a plain launch: after an event wait, programmatic serialization has
    // nothing to overlap (griddepcontrol.wait is then a no-op)
    FF_LAUNCH(K_HEAD_ADAM, (double)kClasses * hd->F * (ha.nrb * 4.0 + 28), hd->side,
              (k_head_adam<<<vblocks + 1, 256, 0, hd->side>>>(ha), cudaGetLastError()), "block Adam");
  }
  FF_TRY(cudaEventRecord(hd->ev_join, hd->side), "event record");
  if (b16) {
    FF_LAUNCH(K_WGRAD_TC, 2.0 * n * N * K, st,
              tc_gemm_wgrad(static_cast<const bf16*>(L->dZ), L->ldN, static_cast<const bf16*>(X), L->ldK, n, N, K,
                            L->dW, K, &L->ds->err, st),
              "weight-gradient GEMM (tcgen05)");
  } else {
    FF_LAUNCH(K_WGRAD_SIMT, 2.0 * n * N * K, st,
              simt_gemm_wgrad(static_cast<const float*>(L->dZ), L->ldN, static_cast<const float*>(X), L->ldK, n, N,
                              K, L->dW, K, st),
              "weight-gradient GEMM (fp32)");
  }
  AdamArgs aa{};
  aa.W = L->W;
  aa.mW = L->mW;
  aa.vW = L->vW;
  aa.dW = L->dW;
  aa.N = N;
  aa.K = K;
  aa.Wb = b16 ? L->Wb : nullptr;
  aa.ldb = L->ldK;
  aa.b = L->b;
  aa.mb = L->mb;
  aa.vb = L->vb;
  aa.dbpart = L->dbpart;
  aa.nrb = cdiv(n, kPoRows);
  aa.db_out = L->db;
  aa.has_bias = L->cfg.has_bias;
  aa.lr = L->cfg.lr;
  aa.beta1 = L->cfg.beta1;
  aa.beta2 = L->cfg.beta2;
  aa.eps = L->cfg.eps;
  aa.ds = L->ds;
  aa.loss_part = nullptr;
  aa.loss_out = nullptr;
  aa.B = n;
  // data nobody reads after this step (see the FF train step)
  aa.discard_dW = !L->cfg.keep_grad && ((uintptr_t)L->dW & 127u) == 0;
  if (!L->cfg.keep_grad) add_dead(aa, L->dZ, (size_t)n * L->ldN * (size_t)es);
  FF_LAUNCH(K_ADAM, (double)N * K * (28.0 + (b16 ? 2.0 : 0.0)), st, launch_adam(aa, st), "layer Adam");
  FF_TRY(cudaStreamWaitEvent(st, hd->ev_join, 0), "stream wait");
  return FF_OK;
}

ff_status ff_po_predict(ff_layer* const* layers, int n_layers, ff_head* hd, const float* x, int n, int* pred,
                        float* logits, void* stream) {
  ff::NvtxRange nvtx_("ff_po_predict");
  if (!layers || n_layers < 1 || n_layers > kMaxSegs + 1 || !hd || n < 0) return FF_ERR_INVALID_ARG;
  for (int k = 0; k < n_layers; ++k) {
    if (!layers[k]) return FF_ERR_INVALID_ARG;
    if (layers[k]->is_bf16 != layers[0]->is_bf16) return FF_ERR_INVALID_ARG;
    if (k > 0 && layers[k]->K != layers[k - 1]->N) return FF_ERR_INVALID_ARG;
  }
  if (layers[0]->K < kClasses || hd->F != layers[n_layers - 1]->N) return FF_ERR_INVALID_ARG;
  if (n == 0) return FF_OK;
  if (!x || (!pred && !logits)) return FF_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int C = n < hd->cfg.max_rows ? n : hd->cfg.max_rows;
  HeadWork w;
  ff_status s = head_workspace(hd, layers, n_layers, C, false, &w);
  if (s != FF_OK) return s;
  hd->last_stream = st;
  int* err = &hd->ds->err;
  const bool b16 = layers[0]->is_bf16;
  ff_layer* top = layers[n_layers - 1];
  for (int r0 = 0; r0 < n; r0 += C) {
    const int cn = (n - r0) < C ? (n - r0) : C;
    s = head_forward(layers, n_layers, x + (size_t)r0 * layers[0]->K, cn, w, err, st, true);
    if (s != FF_OK) return s;
    Segs sg{};
    sg.H[0] = w.Hk[n_layers - 1];
    sg.s[0] = nullptr;
    sg.ld[0] = top->ldN;
    sg.F[0] = top->N;
    sg.nseg = 1;
    sg.F_total = top->N;
    float* z = logits ? logits + (size_t)r0 * kClasses : w.logits;
    s = head_logits(hd, sg, b16, cn, nullptr, z, w.zpart, nullptr, nullptr, err, st);
    if (s != FF_OK) return s;
    if (pred)
      FF_LAUNCH(K_ARGMAX, (double)cn * 44, st, launch_argmax(z, cn, nullptr, pred + r0, st), "block argmax");
  }
  return FF_OK;
}

}  // extern "C"
