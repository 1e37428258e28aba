// fp32 GEMMs of the FF layer step on the CUDA cores (FFMA), for the exact
// fp32 mode: the same contracts as the tensor-core GEMMs (forward with the
// scale/bias/ReLU/goodness epilogue, plain fp32 store, weight gradient over
// the batch rows), so the fp32 path is the full-precision statement of §3/§4
// on the GPU.  A 128x128 tile per 256-thread CTA, 8x8 outputs per thread,
// K in steps of 8 through double-buffered shared memory.  A GEMM of few
// tiles (the 128-row steps of a small batch: 4 CTAs for 128 x 500) is
// latency-bound on its long K loop, so it splits K over up to 8 CTAs per
// tile: each writes its partial tile, and the last to arrive (an arrival
// counter per tile, no waiting) adds the partials in split order and runs
// the epilogue.
#include "ff_internal.cuh"

namespace ff {
namespace {

constexpr int TM = 128, TN = 128, TK = 8, NT = 256;
constexpr int MODE_FWD = 0, MODE_STORE = 1;
constexpr int kMaxSplit = 8;
constexpr int kSplitBelow = 76;  // split GEMMs of fewer tiles than half the SMs

int split_of(int M, int N, int K) {
  const int tiles = cdiv(N, TN) * cdiv(M, TM);
  const int steps = cdiv(K, TK);
  if (tiles >= kSplitBelow || steps < 16) return 1;
  int S = cdiv(kSplitBelow, tiles);
  if (S > kMaxSplit) S = kMaxSplit;
  if (S > steps / 4) S = steps / 4;  // at least 4 K steps per split
  return S < 1 ? 1 : S;
}

// Loads the TK x 128 slice [k0, k0+TK) of an operand whose tile rows start
// at r0.  MN == false: element (r, k) at P[r * ld + k]; MN == true: at
// P[k * ld + r].  Out-of-range elements read as zero.
template <bool MN>
__device__ __forceinline__ void load_tile(const float* __restrict__ P, int ld, int rows, int K, int r0, int k0,
                                          float (&v)[4]) {
  const int tid = threadIdx.x;
  if (!MN) {
    const int r = r0 + tid / 2, k = k0 + (tid & 1) * 4;
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = (r < rows && k + u < K) ? __ldg(P + (size_t)r * ld + k + u) : 0.f;
  } else {
    const int k = k0 + tid / 32, r = r0 + (tid & 31) * 4;
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = (k < K && r + u < rows) ? __ldg(P + (size_t)k * ld + r + u) : 0.f;
  }
}

template <bool MN>
__device__ __forceinline__ void store_tile(float (*S)[TM + 4], const float (&v)[4]) {
  const int tid = threadIdx.x;
  if (!MN) {
    const int r = tid / 2, k = (tid & 1) * 4;
#pragma unroll
    for (int u = 0; u < 4; ++u) S[k + u][r] = v[u];
  } else {
    const int k = tid / 32, r = (tid & 31) * 4;
    *reinterpret_cast<float4*>(&S[k][r]) = make_float4(v[0], v[1], v[2], v[3]);
  }
}

template <bool A_MN, bool B_MN, int MODE>
__global__ void __launch_bounds__(NT) k_simt_gemm(const float* __restrict__ A, int lda, const float* __restrict__ B,
                                                  int ldb, int M, int N, int K, EpiArgs ep) {
  __shared__ __align__(16) float As[2][TK][TM + 4];
  __shared__ __align__(16) float Bs[2][TK][TN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.y * TM, n0 = blockIdx.x * TN;
  // this CTA's share of K: split blockIdx.z of gridDim.z (whole TK steps)
  const int S = gridDim.z;
  const int per = ((K + TK - 1) / TK + S - 1) / S;
  const int kb = blockIdx.z * per * TK;
  const int ke = min(K, kb + per * TK);

  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

  float ra[4], rb[4];
  load_tile<A_MN>(A, lda, M, K, m0, kb, ra);
  load_tile<B_MN>(B, ldb, N, K, n0, kb, rb);
  store_tile<A_MN>(As[0], ra);
  store_tile<B_MN>(Bs[0], rb);
  __syncthreads();

  for (int k0 = kb; k0 < ke; k0 += TK) {
    const int buf = ((k0 - kb) / TK) & 1;
    const bool more = k0 + TK < ke;
    if (more) {
      load_tile<A_MN>(A, lda, M, K, m0, k0 + TK, ra);
      load_tile<B_MN>(B, ldb, N, K, n0, k0 + TK, rb);
    }
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][k][ty * 4]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][k][64 + ty * 4]);
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[buf][k][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[buf][k][64 + tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) {
      store_tile<A_MN>(As[buf ^ 1], ra);
      store_tile<B_MN>(Bs[buf ^ 1], rb);
    }
    __syncthreads();
  }

  if (S > 1) {
    // partial tile out (each thread its own 64 values), then the last CTA of
    // the tile adds the S partials in split order
    const int tile = blockIdx.y * gridDim.x + blockIdx.x;
    const size_t ntile = (size_t)gridDim.x * gridDim.y;
    float* mine = ep.kpart + ((size_t)blockIdx.z * ntile + tile) * (TM * TN) + threadIdx.x * 64;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      *reinterpret_cast<float4*>(mine + i * 8) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
      *reinterpret_cast<float4*>(mine + i * 8 + 4) = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
    }
    __shared__ int last;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(ep.kcnt + tile, 1) == S - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    if (threadIdx.x == 0) ep.kcnt[tile] = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
    for (int z = 0; z < S; ++z) {
      const float* p = ep.kpart + ((size_t)z * ntile + tile) * (TM * TN) + threadIdx.x * 64;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float4 u = __ldcg(reinterpret_cast<const float4*>(p + i * 8));
        const float4 v = __ldcg(reinterpret_cast<const float4*>(p + i * 8 + 4));
        acc[i][0] += u.x; acc[i][1] += u.y; acc[i][2] += u.z; acc[i][3] += u.w;
        acc[i][4] += v.x; acc[i][5] += v.y; acc[i][6] += v.z; acc[i][7] += v.w;
      }
    }
  }

#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int gi = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
    if (MODE == MODE_FWD) {
      float g = 0.f;
      if (gi < M) {
        const float s = ep.row_scale[gi];
        float* out = reinterpret_cast<float*>(ep.out) + (size_t)gi * ep.ldo;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int col = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
          float h = 0.f;
          if (col < N) {
            float z = s * acc[i][j];
            if (ep.bias) z += __ldg(ep.bias + col);
            h = z != z ? z : fmaxf(z, 0.f);  // ReLU, NaN kept for the non-finite check
          }
          g = fmaf(h, h, g);
          if (col < ep.ldo) out[col] = h;
        }
      }
      // the 16 threads sharing this row are lanes tx = 0..15 of one half-warp
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
      if (tx == 0 && gi < M) ep.gpart[(size_t)blockIdx.x * M + gi] = g;
    } else {
      if (gi < M) {
        float* out = reinterpret_cast<float*>(ep.out) + (size_t)gi * ep.ldo;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int col = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + (j - 4));
          if (col < N) out[col] = acc[i][j];
        }
      }
    }
  }
}

template <bool A_MN, bool B_MN, int MODE>
cudaError_t launch(const float* A, int lda, const float* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                   cudaStream_t st) {
  const int tiles = cdiv(N, TN) * cdiv(M, TM);
  int S = ep.kpart && ep.kcnt ? split_of(M, N, K) : 1;
  if (S > 1 && ((size_t)S * tiles * TM * TN > ep.kpart_cap || tiles > ep.kcnt_cap)) S = 1;
  dim3 grid(cdiv(N, TN), cdiv(M, TM), S);
  k_simt_gemm<A_MN, B_MN, MODE><<<grid, NT, 0, st>>>(A, lda, B, ldb, M, N, K, ep);
  return cudaGetLastError();
}

}  // namespace

int simt_fwd_ntiles(int N) { return cdiv(N, TN); }
size_t simt_split_floats(int M, int N, int K) {
  const int S = split_of(M, N, K);
  return S > 1 ? (size_t)S * cdiv(N, TN) * cdiv(M, TM) * TM * TN : 0;
}
int simt_split_tiles(int M, int N) { return cdiv(N, TN) * cdiv(M, TM); }

cudaError_t simt_gemm_fwd(const float* A, int lda, const float* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                          cudaStream_t st) {
  return launch<false, false, MODE_FWD>(A, lda, B, ldb, M, N, K, ep, st);
}

cudaError_t simt_gemm_store(const float* A, int lda, const float* B, int ldb, int M, int N, int K, float* C, int ldc,
                            cudaStream_t st) {
  EpiArgs ep{nullptr, nullptr, C, ldc, nullptr};
  return launch<false, false, MODE_STORE>(A, lda, B, ldb, M, N, K, ep, st);
}

cudaError_t simt_gemm_wgrad(const float* G, int ldg, const float* X, int ldx, int R, int N, int K, float* C, int ldc,
                            cudaStream_t st, const EpiArgs* split) {
  // C[N, K] = sum_r G[r, n] X[r, k]: rows of C index G's columns (MN-major A),
  // columns of C index X's columns (MN-major B), contraction over R.
  EpiArgs ep{nullptr, nullptr, C, ldc, nullptr};
  if (split) {
    ep.kpart = split->kpart;
    ep.kpart_cap = split->kpart_cap;
    ep.kcnt = split->kcnt;
    ep.kcnt_cap = split->kcnt_cap;
  }
  return launch<true, true, MODE_STORE>(G, ldg, X, ldx, N, K, R, ep, st);
}

}  // namespace ff
