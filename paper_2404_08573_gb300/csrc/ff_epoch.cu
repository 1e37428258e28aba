// The FF train step of a whole net over many batches in ONE persistent
// kernel (bf16 operands, fp32 accumulation and master weights).
//
// Work.  Batch b is the concatenated positive/negative batch of §4 (2B rows);
// per layer k and batch b the step of §3 (Eq. 1) and §5.1 is cut into tasks:
//   OV(b, 64 rows)        label overlay, cast to bf16, row scale (layer 1 input)
//   FWD(k, b, rt, ct)     256 x 256 tile of H = ReLU(s X W^T + b) with its
//                         per-128-column goodness partials (tcgen05, pair of CTAs)
//   LG(k, b, 64 rows)     goodness, loss, dL/dg, next-layer scale, dZ' = s 2 dL/dg H,
//                         bias-gradient partials
//   WG(k, b, nt, kt)      256 x 256 tile of dW = dZ'^T X (tcgen05, pair of CTAs)
//   ADAM(k, b, 16 rows)   Adam on 16 rows of W and their bias elements; refreshes
//                         the bf16 copy of W; the first chunk also forms the loss
// Layers run as a wavefront: in tick t layer k works on batch t - k, so the
// four layers' tasks of a tick are independent -- the single-GPU analogue of
// Single-Layer PFF (§4.1, Algorithm 1), inside one launch instead of on
// streams.  Every task computes exactly what the per-step kernels compute
// (same tile shapes for the goodness partials, same reduction orders), so an
// epoch here is bitwise equal to the same batches through ff_net_train_step.
//
// Execution.  One CTA per SM, in pairs (clusters of 2 along x).  Each CTA runs
// three roles at once:
//   warp 0        TMA producer (the even CTA's lane 0 also dequeues GEMM tasks
//                 and hands them to both CTAs through a shared-memory ring)
//   warp 1        tcgen05.mma issuer (even CTA), TMEM owner
//   warps 2..5    GEMM epilogue (TMEM -> registers -> TMA stores), with two
//                 256-column accumulators so a tile's epilogue overlaps the
//                 next tile's mainloop
//   warps 6..31   streamers: OV, LG and ADAM tasks (HBM-bound), dequeued one
//                 at a time by the CTA
// So Adam's HBM stream and the local gradient run on every SM beside the
// tensor-core tiles.  Tasks are dequeued in a fixed global order in which
// every dependency points to an earlier task; dependencies are
// monotonically increasing completion counters in global memory, waited on
// with acquire loads and bumped with release reductions.  Every wait is
// bounded (kWaitTimeoutNs): a timeout latches DEVERR_TIMEOUT and an abort flag
// that every role polls, and the CTA winds down (in-flight copies and MMAs
// drained, TMEM freed).
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <vector>

#include "ff_api_internal.h"
#include "ff_net_internal.h"
#include "ff_ptx.cuh"

namespace ff {

namespace {

constexpr int kMaxLayers = 8;
constexpr int kMaxTiles = 64;     // row tiles (2B / 256) and column tiles (N / 256) per layer
constexpr int BM = 128;           // rows each CTA of a pair computes
constexpr int BK = 64;            // one 128-byte swizzle row of bf16
constexpr int BN = 256;           // columns of a pair tile
constexpr int HB = BN / 2;        // B columns each CTA of the pair loads
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = HB * BK * 2;
constexpr int STAGE = A_BYTES + B_BYTES;
constexpr int EPI_WARPS = 4;    // one per TMEM lane quarter, both column halves
constexpr int STR_WARPS = 26;   // 32 warps in all (64 registers a thread): many loads in flight per SM
constexpr int EPI0 = 2;
constexpr int STR0 = EPI0 + EPI_WARPS;
constexpr int NTHREADS = 32 * (STR0 + STR_WARPS);
constexpr int NSTR = 32 * STR_WARPS;  // streamer threads
constexpr int TQ = 4;             // task ring slots between the GEMM roles
constexpr uint32_t TMEM_COLS = 512;  // two 256-column accumulators
constexpr int EPI_BYTES = 16384;  // staging per epilogue warp: its 32 rows x 256 bf16 columns
constexpr int LG_ROWS = 32;      // rows of a bias-gradient partial (as k_grad_prep)
constexpr int LG_TASK_ROWS = 64; // rows of a local-gradient task
constexpr int OV_ROWS = 64;
constexpr int ADAM_ROWS = 16;
constexpr int BAR_EPI = 1, BAR_STR = 2;

constexpr int OFF_EPI = STAGES * STAGE;
constexpr int OFF_BIAS = OFF_EPI + EPI_WARPS * EPI_BYTES;
constexpr int OFF_RED = OFF_BIAS + BN * 4;
constexpr int RED_FLOATS = 4 * LG_TASK_ROWS + 6 * 8 + 2 * 64;  // rows' terms, row-group sums, active counts
constexpr int OFF_BARS = OFF_RED + RED_FLOATS * 4;
// full[STAGES], empty[STAGES], accf[2], acce[2], tqf[TQ], tqe[TQ], drain
constexpr int NBARS = 2 * STAGES + 4 + 2 * TQ + 1;
constexpr int OFF_TQ = OFF_BARS + NBARS * 8;
constexpr int OFF_MISC = OFF_TQ + TQ * 12;
constexpr int SMEM_BYTES = OFF_MISC + 64 + 1024;  // + 1024-byte alignment slack
static_assert(24 + 4 * EPI_WARPS <= 64, "misc slots");
static_assert(SMEM_BYTES <= 227 * 1024, "shared memory per CTA");
static_assert(OFF_EPI % 1024 == 0 && STAGE % 1024 == 0, "swizzled tiles need 1024-byte alignment");

enum : uint32_t { T_FWD = 0, T_WG = 1, T_OV = 2, T_LG = 3, T_ADAM = 4, T_END = 7 };

__host__ __device__ inline uint2 mk_task(uint32_t type, uint32_t k, uint32_t b, uint32_t a, uint32_t c) {
  return make_uint2(type | (k << 3) | (b << 6), a | (c << 16));
}

// Completion counters (ints, zero at launch).
constexpr int C_QG = 0, C_QS = 1, C_ABORT = 2;
constexpr int C_BASE = 32;
__host__ __device__ constexpr int c_fwd(int k, int rt) { return C_BASE + (0 * kMaxLayers + k) * kMaxTiles + rt; }
__host__ __device__ constexpr int c_lgrt(int k, int rt) { return C_BASE + (1 * kMaxLayers + k) * kMaxTiles + rt; }
__host__ __device__ constexpr int c_wgnt(int k, int nt) { return C_BASE + (2 * kMaxLayers + k) * kMaxTiles + nt; }
__host__ __device__ constexpr int c_adam(int k, int nt) { return C_BASE + (3 * kMaxLayers + k) * kMaxTiles + nt; }
__host__ __device__ constexpr int c_lgall(int k) { return C_BASE + 4 * kMaxLayers * kMaxTiles + k; }
__host__ __device__ constexpr int c_wgall(int k) { return C_BASE + 4 * kMaxLayers * kMaxTiles + kMaxLayers + k; }
// Overlay blocks are counted per ring slot: the overlays of consecutive
// batches do not wait for each other, so a count over all batches could reach
// batch b's target while a block of b is still unwritten; the writes of one
// slot are ordered (the overlay of b + D waits for the readers of b).
constexpr int kMaxSlots = 64;
__host__ __device__ constexpr int c_ov(int slot, int rt) {
  return C_BASE + 4 * kMaxLayers * kMaxTiles + 2 * kMaxLayers + slot * kMaxTiles + rt;
}
constexpr int N_COUNTERS = C_BASE + 4 * kMaxLayers * kMaxTiles + 2 * kMaxLayers + kMaxSlots * kMaxTiles;

// Tensor maps of a layer (in global memory).
enum { TM_FWD_A = 0, TM_FWD_B, TM_FWD_C, TM_WG_A, TM_WG_B, TM_WG_C, TM_N };

struct LayerP {
  int K, N, ldK, ldN;
  int n_ct;                 // 256-column tiles of H (= 256-row tiles of dW)
  int n_kt;                 // 256-column tiles of dW
  int n_chunks;             // Adam chunks of ADAM_ROWS rows
  int has_bias, discard_dW;
  float theta, lr, beta1, beta2, eps;
  double beta1d, beta2d;
  const float* s_in_ring;   // [D * M] row scale of this layer's input rows
  bf16* h_ring;             // [D * M, ldN] activity
  float* g_ring;            // [D][2 * n_ct][M] goodness partials
  float* sn_ring;           // [D * M] next layer's row scale (null for the last layer)
  bf16* dZ;                 // [M, ldN] weight-gradient operand s * dZ
  float* dW;                // [N, K]
  float *W, *mW, *vW, *b, *mb, *vb, *db_out;
  bf16* Wb;                 // [N, ldK]
  float *dbpart, *loss_part, *stat_part;
  ff_dev_state* ds;
  const CUtensorMap* tm;    // [TM_N]
};

struct EpochP {
  int L, D, M, B, nb, xrp, K0, ldK0;
  const float* x;           // images: xrp rows per pair (2: the stacked pair batches; 1: one image per pair)
  const int* labels;        // [nb * M]
  bf16* x0_ring;            // [D * M, ldK0] layer-1 input
  float* s0_ring;           // [D * M]
  const uint2* gtask;
  int n_gtask;
  const uint2* stask;
  int n_stask;
  int* cnt;
  int* err;
  float* loss;              // [nb, L] or null
  // optional trace: per task (GEMM tasks first, then stream tasks) its
  // dequeue, dependencies-met and done times (%globaltimer, ns) and SM id
  unsigned long long* trace;
  // Roles by cluster: clusters 0 .. gemm_clusters-1 take GEMM tasks; with
  // split set they take no stream tasks and the other clusters take only
  // stream tasks (every CTA takes both otherwise).
  int gemm_clusters, split;
  LayerP lay[kMaxLayers];
};

// ------------------------------------------------------------ memory model
__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Orders async-proxy (TMA) accesses of global memory with generic ones.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Starts bringing [p, p + bytes) into L2 (16-byte aligned, in pieces of at
// most 32 KB); nothing waits for it.
__device__ __forceinline__ void prefetch_l2(const void* p, size_t bytes) {
  const char* c = static_cast<const char*>(p);
  for (size_t off = 0; off < bytes; off += 32768) {
    const uint32_t n = (uint32_t)(bytes - off < 32768 ? bytes - off : 32768) & ~15u;
    if (n) asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(c + off), "r"(n) : "memory");
  }
}

__device__ __forceinline__ uint4 ldcg16(const void* p) { return __ldcg(reinterpret_cast<const uint4*>(p)); }

using ptx::mbar_arrive_remote;
using ptx::mbar_try_wait_cluster;
using ptx::st_remote_u1;
using ptx::st_remote_u2;

__device__ __forceinline__ void latch_abort(const EpochP& P) {
  atomicOr(P.err, DEVERR_TIMEOUT);
  atomicExch(P.cnt + C_ABORT, 1);
}
__device__ __forceinline__ bool aborted(const EpochP& P) {
  return *reinterpret_cast<volatile const int*>(P.cnt + C_ABORT) != 0;
}

// Bounded wait on an mbarrier phase (cluster-scope acquire); false on abort
// or timeout (the latter latched).  The abort flag lives in global memory, so
// it is read only every 64th poll: a read in every poll would put an L2
// round trip between a phase completing and the waiter seeing it.
__device__ bool bar_wait(const EpochP& P, uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = ptx::globaltimer();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((n & 63u) == 0) {
      if (aborted(P)) return false;
      if (ptx::globaltimer() - t0 > kWaitTimeoutNs) {
        latch_abort(P);
        return false;
      }
    }
  }
}
// Waits, ignoring the abort flag, up to timeout_ns (drains after an abort).
__device__ void bar_drain(uint64_t* bar, uint32_t parity, unsigned long long timeout_ns) {
  const uint64_t t0 = ptx::globaltimer();
  while (!mbar_try_wait_cluster(bar, parity))
    if (ptx::globaltimer() - t0 > timeout_ns) return;
}
// Bounded wait until counter >= target (the abort flag read every 16th poll).
__device__ bool wait_count(const EpochP& P, int idx, int target) {
  const int* p = P.cnt + idx;
  if (ld_acquire(p) >= target) return true;
  const uint64_t t0 = ptx::globaltimer();
  for (uint32_t n = 1;; ++n) {
    if (ld_acquire(p) >= target) return true;
    if ((n & 15u) == 0) {
      if (aborted(P)) return false;
      if (ptx::globaltimer() - t0 > kWaitTimeoutNs) {
        latch_abort(P);
        return false;
      }
    }
  }
}

__device__ __forceinline__ uint32_t smid() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
  return r;
}
// Trace words per task: GEMM tasks -- 0 dequeued, 1 dependencies met
// (producer), 2 MMAs started, 3 last MMA issued, 4 epilogue started, 5 done;
// stream tasks -- 0 dequeued, 1 dependencies met, 5 done; word 2 of a
// stream task is its SM.
}  // namespace
constexpr int kTraceWords = 6;
namespace {
__device__ __forceinline__ void trace_at(const EpochP& P, int idx, int field) {
  if (P.trace) P.trace[(size_t)idx * kTraceWords + field] = ptx::globaltimer();
}
__device__ __forceinline__ void trace_sm(const EpochP& P, int idx) {
  if (P.trace) P.trace[(size_t)idx * kTraceWords + 2] = smid();
}

__device__ __forceinline__ uint32_t t_type(uint2 t) { return t.x & 7u; }
__device__ __forceinline__ int t_layer(uint2 t) { return (int)((t.x >> 3) & 7u); }
__device__ __forceinline__ int t_batch(uint2 t) { return (int)(t.x >> 6); }
__device__ __forceinline__ int t_a(uint2 t) { return (int)(t.y & 0xFFFFu); }
__device__ __forceinline__ int t_c(uint2 t) { return (int)(t.y >> 16); }

__device__ __forceinline__ int chunks_in_tile(const LayerP& lp, int nt) {
  const int rows = lp.N - nt * BN < BN ? lp.N - nt * BN : BN;
  return (rows + ADAM_ROWS - 1) / ADAM_ROWS;
}

// Everything a task reads must be complete, and everything it overwrites
// must have been read by its earlier readers.  Only the dependencies that do
// not already follow from these through the chain
//   FWD(k,b) -> LG(k,b) -> WG(k,b) -> ADAM(k,b) -> FWD(k,b+1)
// are listed.
__device__ bool wait_deps(const EpochP& P, uint2 t) {
  const int k = t_layer(t), b = t_batch(t), a = t_a(t), c = t_c(t);
  switch (t_type(t)) {
    case T_FWD: {
      const LayerP& lp = P.lay[k];
      // the input rows of this row tile, and their row scale
      if (k == 0) {
        if (!wait_count(P, c_ov(b % P.D, a), (BN / OV_ROWS) * (b / P.D + 1))) return false;
      } else if (!wait_count(P, c_lgrt(k - 1, a), (BN / LG_TASK_ROWS) * (b + 1))) {
        return false;
      }
      // this column tile's rows of W and b after the previous batch's update
      if (b >= 1 && !wait_count(P, c_adam(k, c), b * chunks_in_tile(lp, c))) return false;
      // the activity ring slot: the next layer's weight gradient of batch b - D read it
      if (k + 1 < P.L && b >= P.D) {
        const LayerP& ln = P.lay[k + 1];
        if (!wait_count(P, c_wgall(k + 1), (b - P.D + 1) * 2 * ln.n_ct * ln.n_kt)) return false;
      }
      return true;
    }
    case T_WG:
      return wait_count(P, c_lgall(k), (b + 1) * (P.M / LG_TASK_ROWS));
    case T_OV:
      if (b >= P.D) {
        const LayerP& l0 = P.lay[0];
        return wait_count(P, c_wgall(0), (b - P.D + 1) * 2 * l0.n_ct * l0.n_kt);
      }
      return true;
    case T_LG:
      return wait_count(P, c_fwd(k, a / (BN / LG_TASK_ROWS)), (b + 1) * 2 * P.lay[k].n_ct);
    case T_ADAM:
      return wait_count(P, c_wgnt(k, a * ADAM_ROWS / BN), (b + 1) * 2 * P.lay[k].n_kt);
  }
  return true;
}

__device__ void signal_done(const EpochP& P, uint2 t) {
  const int k = t_layer(t), a = t_a(t);
  switch (t_type(t)) {
    case T_FWD: red_release_add(P.cnt + c_fwd(k, a), 1); break;
    case T_WG:
      red_release_add(P.cnt + c_wgnt(k, a), 1);
      red_release_add(P.cnt + c_wgall(k), 1);
      break;
    case T_OV: red_release_add(P.cnt + c_ov(t_batch(t) % P.D, a / (BN / OV_ROWS)), 1); break;
    case T_LG:
      red_release_add(P.cnt + c_lgrt(k, a / (BN / LG_TASK_ROWS)), 1);
      red_release_add(P.cnt + c_lgall(k), 1);
      break;
    case T_ADAM: red_release_add(P.cnt + c_adam(k, a * ADAM_ROWS / BN), 1); break;
  }
}


// ------------------------------------------------------------- stream tasks
// s: streamer thread 0..NSTR-1 (s >> 5 its warp, lane its lane).

// OV(b, r64): the label overlay of §3 for 64 rows of batch b, as k_overlay
// (mode 0): features 0..9 <- one-hot(label), bf16 cast, row scale.  A warp
// takes a row; all of a lane's loads of the row are issued before its first
// store (the row scale sums each lane's values in k_overlay's order).
constexpr int OV_VEC_MAX = 8;  // float4 loads per lane and row: rows up to 4096 features
__device__ __noinline__ void task_overlay(const EpochP& P, int b, int r64, int s) {
  const int y = s >> 5, lane = s & 31;
  const int F = P.K0, ldo = P.ldK0, slot = b % P.D;
  const bool vec = (F & 3) == 0 && (reinterpret_cast<uintptr_t>(P.x) & 15u) == 0 && ldo <= 128 * OV_VEC_MAX;
  for (int rr = y; rr < OV_ROWS; rr += STR_WARPS) {
    const int row = r64 * OV_ROWS + rr;
    const float* xr = P.xrp == 2 ? P.x + ((size_t)b * P.M + row) * F : P.x + ((size_t)b * P.B + row % P.B) * F;
    bf16* orow = P.x0_ring + ((size_t)slot * P.M + row) * ldo;
    const int lab = __ldg(P.labels + (size_t)b * P.M + row);
    float ss = 0.f;
    if (vec) {
      float4 q[OV_VEC_MAX];
#pragma unroll
      for (int it = 0; it < OV_VEC_MAX; ++it) {
        const int f = 4 * lane + 128 * it;
        q[it] = f < F ? __ldg(reinterpret_cast<const float4*>(xr + f)) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int it = 0; it < OV_VEC_MAX; ++it) {
        const int f = 4 * lane + 128 * it;
        if (f >= ldo) break;
        float v[4] = {q[it].x, q[it].y, q[it].z, q[it].w};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (f + u < 10) v[u] = (f + u == lab) ? 1.f : 0.f;
          ss = fmaf(v[u], v[u], ss);
        }
        __nv_bfloat162 p0 = __floats2bfloat162_rn(v[0], v[1]), p1 = __floats2bfloat162_rn(v[2], v[3]);
        *reinterpret_cast<uint2*>(orow + f) =
            make_uint2(*reinterpret_cast<uint32_t*>(&p0), *reinterpret_cast<uint32_t*>(&p1));
      }
    } else {
      for (int f = lane; f < ldo; f += 32) {
        float v = 0.f;
        if (f < F) v = (f < 10) ? (f == lab ? 1.f : 0.f) : __ldg(xr + f);
        orow[f] = __float2bfloat16_rn(v);
        ss = fmaf(v, v, ss);
      }
    }
    ss = warp_sum(ss);
    if (lane == 0) P.s0_ring[(size_t)slot * P.M + row] = inv_norm(ss);
  }
}

// LG(k, b, t): the local gradient of rows [64t, 64t + 64) -- two 32-row
// blocks, each what the 256-column blocks of k_grad_prep compute for it, with
// the same reduction orders:
//   1. warps 0..15 (per block, k_grad_prep's 8 row groups ty with 8 lanes per
//      row) sum each row's goodness partials and form dL/dg, the next layer's
//      scale and the row's loss and goodness terms (summed per row group,
//      then over the groups in order);
//   2. every streamer thread takes (block, 8-column chunk) items: dZ' =
//      (s 2 dL/dg) h for the block's 32 rows, and the bias-gradient partial of
//      each column as k_grad_prep sums it (per row group its 4 rows in
//      order, then the 8 groups in order).
__device__ __noinline__ void task_local_grad(const EpochP& P, int k, int b, int t, int s, float* smem_red) {
  const LayerP& lp = P.lay[k];
  const int slot = b % P.D;
  const int M = P.M, N = lp.N, ld = lp.ldN;
  const int ntiles = 2 * lp.n_ct;
  const int nrb = M / LG_ROWS, ncb = (ld + 255) / 256;
  constexpr int NBLK = LG_TASK_ROWS / LG_ROWS;
  const bf16* H = lp.h_ring + (size_t)slot * M * ld;
  const float* gpart = lp.g_ring + (size_t)slot * ntiles * M;
  const float* sin = lp.s_in_ring + (size_t)slot * M;
  float* s_next = lp.sn_ring ? lp.sn_ring + (size_t)slot * M : nullptr;
  float* sc_row = smem_red;                    // [64] s_i * 2 dL/dg_i
  float* c_row = sc_row + LG_TASK_ROWS;        // [64] 2 dL/dg_i
  float* lred = c_row + LG_TASK_ROWS;          // [2][8] per block and row group: loss
  float* gpred = lred + NBLK * 8;              // positive rows' goodness
  float* gnred = gpred + NBLK * 8;             // negative rows' goodness
  int* actc = reinterpret_cast<int*>(gnred + NBLK * 8);  // [2][64] active ReLUs per block and 256-column block
  const int w = s >> 5, lane = s & 31;
  const int r0 = t * LG_TASK_ROWS;
  for (int i = s; i < NBLK * 64; i += NSTR) actc[i] = 0;
  if (w < NBLK * 8) {
    const int blk = w >> 3, ty = w & 7, q = lane >> 3, p = lane & 7;
    const int lr = blk * LG_ROWS + ty + 8 * q;  // row within the task
    const int i = r0 + lr;
    float g = 0.f;
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int tt = p + 8 * u;
      v[u] = tt < ntiles ? __ldcg(gpart + (size_t)tt * M + i) : 0.f;
    }
    for (int tt = p + 64; tt < ntiles; tt += 8) v[0] += __ldcg(gpart + (size_t)tt * M + i);
#pragma unroll
    for (int u = 0; u < 8; ++u) g += v[u];
    g += __shfl_xor_sync(0xffffffffu, g, 4);
    g += __shfl_xor_sync(0xffffffffu, g, 2);
    g += __shfl_xor_sync(0xffffffffu, g, 1);
    float lv = 0.f, gp = 0.f, gn = 0.f;
    if (p == 0) {
      const bool pos = i < P.B;
      const float tt = pos ? lp.theta - g : g - lp.theta;
      const float sg = sigmoid_f(tt);
      const float cc = 2.f * (pos ? -sg : sg) / (float)P.B;
      c_row[lr] = cc;
      sc_row[lr] = __ldcg(sin + i) * cc;
      if (!isfinite(g)) atomicOr(&lp.ds->err, DEVERR_NONFINITE);
      if (s_next) s_next[i] = inv_norm(g);
      lv = softplus_f(tt);
      (pos ? gp : gn) = g;
    }
    lv = warp_sum(lv);
    gp = warp_sum(gp);
    gn = warp_sum(gn);
    if (lane == 0) {
      lred[w] = lv;
      gpred[w] = gp;
      gnred[w] = gn;
    }
  }
  ptx::named_bar(BAR_STR, NSTR);
  if (s < NBLK) {
    const int rb = t * NBLK + s;
    float tl = 0.f, tp = 0.f, tn = 0.f;
#pragma unroll
    for (int yy = 0; yy < 8; ++yy) {
      tl += lred[s * 8 + yy];
      tp += gpred[s * 8 + yy];
      tn += gnred[s * 8 + yy];
    }
    lp.loss_part[rb] = tl;
    lp.stat_part[rb] = tp;
    lp.stat_part[nrb + rb] = tn;
    if (rb == 0) {
      // the Adam update that follows is step t; beta^t kept as running
      // products (read around L1: other SMs wrote them earlier in this launch)
      ff_dev_state* ds = lp.ds;
      const double p1 = __ldcg(&ds->pow1) * lp.beta1d, p2 = __ldcg(&ds->pow2) * lp.beta2d;
      ds->t = __ldcg(&ds->t) + 1;
      ds->pow1 = p1;
      ds->pow2 = p2;
      ds->bc1 = (float)(1.0 - p1);
      ds->bc2 = (float)(1.0 - p2);
    }
  }
  const int nch = ld / 8;  // 8-column chunks (ld is a multiple of 8)
  for (int item = s; item < NBLK * nch; item += NSTR) {
    const int blk = item / nch, ch = item - blk * nch;
    const int cg = 8 * ch, rb0 = r0 + blk * LG_ROWS, lb = blk * LG_ROWS;
    // row group y holds rows y, y + 8, y + 16, y + 24 of the block (kept
    // packed: 8 bf16 in 4 registers; the many streamer threads keep enough
    // of these loads in flight)
    auto load_group = [&](int y, uint4 (&hv)[4]) {
#pragma unroll
      for (int q = 0; q < 4; ++q) hv[q] = ldcg16(H + (size_t)(rb0 + y + 8 * q) * ld + cg);
    };
    float tsum[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) tsum[e] = 0.f;
    int act = 0;
    auto use_group = [&](int y, const uint4 (&hp)[4]) {
      float acc[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float ck = c_row[lb + y + 8 * q], sk = sc_row[lb + y + 8 * q];
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&hp[q]);
        uint4 outp;
        __nv_bfloat162* o2 = reinterpret_cast<__nv_bfloat162*>(&outp);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(h2[e]);
          acc[2 * e] = fmaf(ck, f.x, acc[2 * e]);
          acc[2 * e + 1] = fmaf(ck, f.y, acc[2 * e + 1]);
          act += (f.x > 0.f ? 1 : 0) + (f.y > 0.f ? 1 : 0);
          o2[e] = __floats2bfloat162_rn(sk * f.x, sk * f.y);
        }
        *reinterpret_cast<uint4*>(lp.dZ + (size_t)(rb0 + y + 8 * q) * ld + cg) = outp;
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) tsum[e] += acc[e];
    };
#pragma unroll 1
    for (int y = 0; y < 8; ++y) {
      uint4 hv[4];
      load_group(y, hv);
      use_group(y, hv);
    }
    const int rb = t * NBLK + blk;
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (cg + e < N) lp.dbpart[(size_t)rb * N + cg + e] = tsum[e];
    // active ReLUs per 256-column block: whole counts, exact in any order
    if (act) atomicAdd(&actc[blk * 64 + ch / 32], act);
  }
  ptx::named_bar(BAR_STR, NSTR);
  for (int i = s; i < NBLK * ncb; i += NSTR) {
    const int blk = i / ncb, cb = i - blk * ncb;
    lp.stat_part[2 * nrb + (size_t)(t * NBLK + blk) * ncb + cb] = (float)actc[blk * 64 + cb];
  }
}

// Eight floats (32 bytes, 32-byte aligned) read once: not kept in L1,
// evicted first from L2.
__device__ __forceinline__ void ld_stream8(const float* p, float (&v)[8]) {
  uint32_t r[8];
  asm volatile("ld.global.L1::no_allocate.L2::evict_first.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "l"(p)
               : "memory");
#pragma unroll
  for (int e = 0; e < 8; ++e) v[e] = __uint_as_float(r[e]);
}
__device__ __forceinline__ void st_stream8(float* p, const float (&v)[8]) {
  __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
  __stcs(reinterpret_cast<float4*>(p + 4), make_float4(v[4], v[5], v[6], v[7]));
}

// ADAM(k, b, c): Adam (§5.1) on rows [16c, 16c + 16) of W and of b, as k_adam
// does it element by element (same bias-gradient reduction order); chunk 0
// also forms the step's loss and statistics.
__device__ __noinline__ void task_adam(const EpochP& P, int k, int b, int c, int s) {
  const LayerP& lp = P.lay[k];
  const int K = lp.K, N = lp.N;
  const int n0 = c * ADAM_ROWS, n1 = n0 + ADAM_ROWS < N ? n0 + ADAM_ROWS : N;
  const float bc1 = __ldcg(&lp.ds->bc1), bc2 = __ldcg(&lp.ds->bc2);
  const float a1 = lp.lr / bc1, r2 = 1.f / bc2;
  const long long base = (long long)n0 * K, end = (long long)n1 * K;
  const long long total = (long long)N * K;
  // 8 parameters per thread and array per step (K % 8 == 0: every chunk
  // starts and ends on 8)
  constexpr int U = 1;
  for (long long q0 = base / 8 + s; q0 * 8 < end; q0 += NSTR * U) {
    float w[U][8], m[U][8], v[U][8], g[U][8];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const long long idx = (q0 + NSTR * u) * 8;
      if (idx < end) {
        ld_stream8(lp.W + idx, w[u]);
        ld_stream8(lp.mW + idx, m[u]);
        ld_stream8(lp.vW + idx, v[u]);
        ld_stream8(lp.dW + idx, g[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const long long idx = (q0 + NSTR * u) * 8;
      if (idx >= end) continue;
#pragma unroll
      for (int e = 0; e < 8; ++e) adam1(w[u][e], m[u][e], v[u][e], g[u][e], a1, lp.beta1, lp.beta2, lp.eps, r2);
      st_stream8(lp.W + idx, w[u]);
      st_stream8(lp.mW + idx, m[u]);
      st_stream8(lp.vW + idx, v[u]);
      // dW of these rows is dead once read: the first of every 4 threads
      // drops the 128-byte line the 4 just read instead of writing it back
      if (lp.discard_dW && (s & 3) == 0 && idx + 32 <= end && idx + 32 <= total) ptx::discard_l2(lp.dW + idx);
      uint4 pk;
      __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&pk);
#pragma unroll
      for (int e = 0; e < 4; ++e) h2[e] = __floats2bfloat162_rn(w[u][2 * e], w[u][2 * e + 1]);
      *reinterpret_cast<uint4*>(lp.Wb + idx) = pk;
    }
  }
  const int nrb = P.M / LG_ROWS;
  const int j = n0 + s;
  if (s < ADAM_ROWS && j < n1) {
    // the bias gradient: row blocks summed in k_adam's order (8 warp sums of
    // every eighth block, batched by 8, then the 8 sums in order)
    float part[8];
#pragma unroll
    for (int w8 = 0; w8 < 8; ++w8) {
      float acc = 0.f;
      for (int rb0 = w8; rb0 < nrb; rb0 += 64) {
        float vv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int rbi = rb0 + 8 * u;
          vv[u] = rbi < nrb ? __ldcg(lp.dbpart + (size_t)rbi * N + j) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) acc += vv[u];
      }
      part[w8] = acc;
    }
    float db = 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u) db += part[u];
    lp.db_out[j] = db;
    if (lp.has_bias) {
      float bb = __ldcg(lp.b + j), mm = __ldcg(lp.mb + j), vv = __ldcg(lp.vb + j);
      adam1(bb, mm, vv, db, a1, lp.beta1, lp.beta2, lp.eps, r2);
      lp.b[j] = bb;
      lp.mb[j] = mm;
      lp.vb[j] = vv;
    }
  }
  if (c == 0) {
    const int w = s >> 5, lane = s & 31;
    if (w == 1) {
      float tot = 0.f;
      for (int rbi = lane; rbi < nrb; rbi += 32) tot += __ldcg(lp.loss_part + rbi);
      tot = warp_sum(tot);
      if (lane == 0) {
        float* out = P.loss ? P.loss + (size_t)b * P.L + k : &lp.ds->loss;
        *out = tot / (float)P.B;
      }
    }
    if (w >= 2 && w <= 4) {
      const int ncb = (lp.ldN + 255) / 256;
      const int n = w == 4 ? nrb * ncb : nrb;
      const float* src = lp.stat_part + (w == 2 ? 0 : w == 3 ? nrb : 2 * nrb);
      float tot = 0.f;
      for (int q = lane; q < n; q += 32) tot += __ldcg(src + q);
      tot = warp_sum(tot);
      if (lane == 0)
        lp.ds->stats[w - 2] = w == 4 ? tot / (2.f * (float)P.B * (float)N) : tot / (float)P.B;
    }
  }
}

// -------------------------------------------------------------- the kernel
__global__ void __launch_bounds__(NTHREADS, 1) k_epoch(const __grid_constant__ EpochP P) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_s = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + OFF_BARS);
  uint64_t* empty = full + STAGES;
  uint64_t* accf = empty + STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* tqf = acce + 2;
  uint64_t* tqe = tqf + TQ;
  uint64_t* drain = tqe + TQ;
  uint2* tq = reinterpret_cast<uint2*>(smem + OFF_TQ);
  int* tqi = reinterpret_cast<int*>(smem + OFF_TQ + TQ * 8);  // [TQ] the tasks' indices (trace)
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  uint2* stask_slot = reinterpret_cast<uint2*>(smem + OFF_MISC + 8);
  volatile int* evote = reinterpret_cast<volatile int*>(smem + OFF_MISC + 24);  // [EPI_WARPS]
  float* sbias = reinterpret_cast<float*>(smem + OFF_BIAS);
  float* sred = reinterpret_cast<float*>(smem + OFF_RED);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = ptx::cluster_ctarank();
  const bool even = crank == 0;
  constexpr uint16_t pmask = 3;
  const bool gemm_cta = (int)(blockIdx.x / 2) < P.gemm_clusters;
  const bool stream_cta = !P.split || !gemm_cta;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      ptx::mbar_init(&accf[i], 1);
      ptx::mbar_init(&acce[i], 2 * EPI_WARPS);
    }
    for (int j = 0; j < TQ; ++j) {
      ptx::mbar_init(&tqf[j], 1);
      ptx::mbar_init(&tqe[j], 2 + 2 * EPI_WARPS);  // even MMA, odd producer, 8 epilogue warps of each CTA
    }
    ptx::mbar_init(drain, 1);
    ptx::fence_mbar_init();
  }
  if (warp == 1) {
    ptx::tmem_alloc_pair(tslot, TMEM_COLS);
    ptx::tmem_relinquish_pair();
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::cluster_sync();
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp == 0) {
    // ------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t full0 = ptx::mapa_shared(ptx::smem_u32(&full[0]), 0u);
      int it = 0, issued_hi = 0;
      for (int i = 0;; ++i) {
        const int j = i % TQ;
        const uint32_t ph = (uint32_t)(i / TQ) & 1u;
        uint2 task;
        if (even) {
          if (!bar_wait(P, &tqe[j], ph ^ 1u)) break;
          // a cluster without the GEMM role hands its roles the end at once
          const int idx = gemm_cta ? atomicAdd(P.cnt + C_QG, 1) : P.n_gtask;
          task = idx < P.n_gtask ? __ldg(P.gtask + idx) : make_uint2(T_END, 0u);
          if (idx < P.n_gtask) {
            trace_at(P, idx, 0);
            tqi[j] = idx;
            st_remote_u1(&tqi[j], 1u, idx);
          }
          tq[j] = task;
          st_remote_u2(&tq[j], 1u, task);
          ptx::mbar_arrive(&tqf[j]);
          mbar_arrive_remote(&tqf[j], 1u);
        } else {
          if (!bar_wait(P, &tqf[j], ph)) break;
          task = tq[j];
          mbar_arrive_remote(&tqe[j], 0u);
        }
        if (t_type(task) == T_END) break;
        if (!wait_deps(P, task)) break;
        if (even) trace_at(P, tqi[j], 1);
        fence_proxy_async_global();
        const int k = t_layer(task), b = t_batch(task), a = t_a(task), c = t_c(task);
        const LayerP& lp = P.lay[k];
        const int slot = b % P.D;
        const bool fwd = t_type(task) == T_FWD;
        const int nkb = fwd ? (lp.K + BK - 1) / BK : P.M / BK;
        const CUtensorMap* mA = lp.tm + (fwd ? TM_FWD_A : TM_WG_A);
        const CUtensorMap* mB = lp.tm + (fwd ? TM_FWD_B : TM_WG_B);
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t sph = (uint32_t)(it / STAGES) & 1u;
          if (!bar_wait(P, &empty[s], sph ^ 1u)) {
            ok = false;
            break;
          }
          if (even) ptx::mbar_arrive_expect_tx(&full[s], 2 * STAGE);
          uint8_t* sa = smem + s * STAGE;
          uint8_t* sb = sa + A_BYTES;
          const uint32_t fb = full0 + 8u * (uint32_t)s;
          const int k0 = kb * BK;
          if (fwd) {
            // A: this CTA's 128 input rows (K-major); B: its half of the tile's W rows
            ptx::tma_load_2d_pair(sa, mA, fb, k0, slot * P.M + a * BN + (int)crank * BM);
            ptx::tma_load_2d_pair(sb, mB, fb, k0, c * BN + (int)crank * HB);
          } else {
            // A: dZ' columns = this CTA's 128 rows of dW (MN-major); B: its half of X's columns
#pragma unroll
            for (int q = 0; q < BM / 64; ++q)
              ptx::tma_load_2d_pair(sa + q * 64 * BK * 2, mA, fb, a * BN + (int)crank * BM + 64 * q, k0);
#pragma unroll
            for (int q = 0; q < HB / 64; ++q)
              ptx::tma_load_2d_pair(sb + q * 64 * BK * 2, mB, fb, c * BN + (int)crank * HB + 64 * q,
                                    slot * P.M + k0);
          }
          issued_hi = it + 1;
        }
        if (!ok) break;
      }
      if (!aborted(P)) {
        // producer tail: the commits of the last stages have arrived, so that
        // no arrival from the other CTA targets this one after it exits
        for (int q = it; q < it + STAGES; ++q)
          if (!bar_wait(P, &empty[q % STAGES], ((uint32_t)(q / STAGES) & 1u) ^ 1u)) break;
      }
      if (aborted(P)) {
        if (even) {
          int lo = issued_hi - STAGES;
          if (lo < 0) lo = 0;
          for (int q = lo; q < issued_hi; ++q) bar_drain(&full[q % STAGES], (uint32_t)(q / STAGES) & 1u, 10000000ull);
        } else {
          const uint64_t t0 = ptx::globaltimer();
          while (ptx::globaltimer() - t0 < 1000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------- MMA
    if (lane == 0 && even) {
      constexpr uint32_t idesc = ptx::idesc_bf16_f32(2 * BM, BN, 0, 0);
      constexpr uint32_t idesc_mn = ptx::idesc_bf16_f32(2 * BM, BN, 1, 1);
      int it = 0;
      bool issued_any = false;
      for (int i = 0;; ++i) {
        const int j = i % TQ;
        if (!bar_wait(P, &tqf[j], (uint32_t)(i / TQ) & 1u)) break;
        const uint2 task = tq[j];
        const int tidx = tqi[j];
        ptx::mbar_arrive(&tqe[j]);
        if (t_type(task) == T_END) break;
        const int buf = i & 1;
        if (!bar_wait(P, &acce[buf], ((uint32_t)(i >> 1) & 1u) ^ 1u)) break;
        ptx::tc_fence_after();
        trace_at(P, tidx, 2);
        const bool fwd = t_type(task) == T_FWD;
        const LayerP& lp = P.lay[t_layer(task)];
        const int nkb = fwd ? (lp.K + BK - 1) / BK : P.M / BK;
        const uint32_t d = tmem + (uint32_t)(buf * BN);
        bool ok = true;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % STAGES;
          if (!bar_wait(P, &full[s], (uint32_t)(it / STAGES) & 1u)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t a_base = ptx::smem_u32(smem + s * STAGE);
          const uint32_t b_base = a_base + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            uint64_t ad, bd;
            if (fwd) {
              ad = ptx::sdesc_sw128(a_base + kk * 32, 16, 1024);
              bd = ptx::sdesc_sw128(b_base + kk * 32, 16, 1024);
            } else {
              ad = ptx::sdesc_sw128(a_base + kk * 2048, 64 * BK * 2, 1024);
              bd = ptx::sdesc_sw128(b_base + kk * 2048, 64 * BK * 2, 1024);
            }
            ptx::umma_f16_pair(d, ad, bd, fwd ? idesc : idesc_mn, (kb | kk) != 0 ? 1u : 0u);
          }
          issued_any = true;
          ptx::umma_commit_pair(&empty[s], pmask);
        }
        if (!ok) break;
        ptx::umma_commit_pair(&accf[buf], pmask);
        trace_at(P, tidx, 3);
      }
      // every MMA issued so far has completed before TMEM can be released
      if (issued_any) {
        ptx::umma_commit_pair(drain, (uint16_t)1);
        bar_drain(drain, 0, 10000000ull);
      }
    }
  } else if (warp < STR0) {
    // ------------------------------------------------------ epilogue
    // Warp w reads TMEM lane quarter q = w % 4 (rows 32q.. of this CTA's 128)
    // over both 128-column halves in turn, each half with its own goodness
    // partial (the per-128-column partials of the per-step forward GEMM).
    const int q = warp & 3;
    const int ew = warp - EPI0;
    uint8_t* stage = smem + OFF_EPI + ew * EPI_BYTES;
    const uint32_t sw = (uint32_t)(lane & 7);
    // Named barriers among the epilogue warps must be reached by all of them
    // or by none: every go/stop decision after a bounded wait is a vote.
    auto vote = [&](bool ok) {
      ok = __all_sync(0xffffffffu, ok);
      if (lane == 0) evote[ew] = ok ? 1 : 0;
      ptx::named_bar(BAR_EPI, 32 * EPI_WARPS);
      bool all = true;
#pragma unroll
      for (int w = 0; w < EPI_WARPS; ++w) all = all && evote[w] != 0;
      ptx::named_bar(BAR_EPI, 32 * EPI_WARPS);  // read before the next vote writes
      return all;
    };
    for (int i = 0;; ++i) {
      const int j = i % TQ;
      const bool got = bar_wait(P, &tqf[j], (uint32_t)(i / TQ) & 1u);
      const uint2 task = got ? tq[j] : make_uint2(T_END, 0u);
      const int tidx = got ? tqi[j] : 0;  // read before the slot is released
      __syncwarp();
      if (got && lane == 0) {
        if (even)
          ptx::mbar_arrive(&tqe[j]);
        else
          mbar_arrive_remote(&tqe[j], 0u);
      }
      // the epilogue's own reads (bias, row scales) and writes follow the
      // same dependencies as the task's operands
      bool ok = got && t_type(task) != T_END;
      if (ok && warp == EPI0 && lane == 0) ok = wait_deps(P, task);
      if (!vote(ok)) break;
      const int k = t_layer(task), b = t_batch(task), a = t_a(task), c = t_c(task);
      const LayerP& lp = P.lay[k];
      const bool fwd = t_type(task) == T_FWD;
      const int slot = b % P.D;
      const int buf = i & 1;
      const int n0 = c * BN;                                  // fwd: first column; wg: first dW column (K)
      const int rloc = a * BN + (int)crank * BM + q * 32;     // this warp's first row (fwd: batch row; wg: dW row)
      float srow = 0.f;
      if (fwd) {
        for (int cc = (int)threadIdx.x - 32 * EPI0; cc < BN; cc += 32 * EPI_WARPS)
          sbias[cc] = (lp.has_bias && n0 + cc < lp.N) ? __ldcg(lp.b + n0 + cc) : 0.f;
        srow = __ldcg(lp.s_in_ring + (size_t)slot * P.M + rloc + lane);
        ptx::named_bar(BAR_EPI, 32 * EPI_WARPS);
      }
      const bool ready = bar_wait(P, &accf[buf], (uint32_t)(i >> 1) & 1u);
      ptx::tc_fence_after();
      if (!vote(ready)) break;
      if (even && warp == EPI0 && lane == 0) trace_at(P, tidx, 4);
      const CUtensorMap* mC = lp.tm + (fwd ? TM_FWD_C : TM_WG_C);
      int fchunk = 0;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        const int cbase = hh * (BN / 2);
        const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN + cbase);
        float g = 0.f;
        if (fwd) {
          // 16 columns at a time (a 16-column TMEM load), the next load in
          // flight while these are used: H = ReLU(s acc + b) to bf16 in the
          // 128-byte-swizzled staging, goodness from the fp32 values in
          // column order
          auto process = [&](const uint32_t (&r)[16], int c0) {
            uint32_t packed[8];
            const float4* b4 = reinterpret_cast<const float4*>(sbias + cbase + c0);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const float4 bb = b4[v];
              const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
              float h[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float z = fmaf(srow, __uint_as_float(r[4 * v + e]), bv[e]);
                h[e] = z != z ? z : fmaxf(z, 0.f);
                g = fmaf(h[e], h[e], g);
              }
              __nv_bfloat162 p0 = __floats2bfloat162_rn(h[0], h[1]);
              __nv_bfloat162 p1 = __floats2bfloat162_rn(h[2], h[3]);
              packed[2 * v] = *reinterpret_cast<uint32_t*>(&p0);
              packed[2 * v + 1] = *reinterpret_cast<uint32_t*>(&p1);
            }
            uint8_t* base = stage + hh * 8192 + (c0 / 64) * (32 * 128) + lane * 128;
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              const uint32_t jj = (uint32_t)((c0 % 64) / 8 + v);
              *reinterpret_cast<uint4*>(base + ((jj ^ sw) << 4)) =
                  make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2], packed[4 * v + 3]);
            }
          };
          uint32_t ra[16], rb[16];
          ptx::tmem_ld16(trow, ra);
          ptx::tmem_ld_wait();
#pragma unroll 1
          for (int c0 = 0; c0 < BN / 2; c0 += 32) {
            ptx::tmem_ld16(trow + (uint32_t)(c0 + 16), rb);
            process(ra, c0);
            ptx::tmem_ld_wait();
            if (c0 + 32 < BN / 2) ptx::tmem_ld16(trow + (uint32_t)(c0 + 32), ra);
            process(rb, c0 + 16);
            ptx::tmem_ld_wait();
            if (c0 % 64 == 32) {
              // a full 64-column box: out to the activity ring
              ptx::fence_async_smem();
              __syncwarp();
              const int col = n0 + cbase + c0 - 32;
              if (lane == 0) {
                if (col < lp.ldN) ptx::tma_store_2d(mC, stage + hh * 8192 + (c0 / 64) * (32 * 128), col, slot * P.M + rloc);
                ptx::bulk_commit();
              }
            }
          }
        } else {
          // fp32 dW, 32 columns (one 4 KB box) at a time through slot n & 1,
          // refilled once the store issued from it two boxes ago has read it
#pragma unroll 1
          for (int c0 = 0; c0 < BN / 2; c0 += 32) {
            uint32_t ra[16], rb[16];
            ptx::tmem_ld16(trow + (uint32_t)c0, ra);
            ptx::tmem_ld16(trow + (uint32_t)(c0 + 16), rb);
            uint8_t* sbuf = stage + (fchunk & 1) * 4096;
            if (lane == 0 && fchunk >= 2) ptx::bulk_wait_read1();
            __syncwarp();
            ptx::tmem_ld_wait();
            uint8_t* base = sbuf + lane * 128;
#pragma unroll
            for (int v = 0; v < 4; ++v)
              *reinterpret_cast<uint4*>(base + (((uint32_t)v ^ sw) << 4)) =
                  make_uint4(ra[4 * v], ra[4 * v + 1], ra[4 * v + 2], ra[4 * v + 3]);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              *reinterpret_cast<uint4*>(base + (((uint32_t)(v + 4) ^ sw) << 4)) =
                  make_uint4(rb[4 * v], rb[4 * v + 1], rb[4 * v + 2], rb[4 * v + 3]);
            ptx::fence_async_smem();
            __syncwarp();
            const int col0 = n0 + cbase + c0;
            if (lane == 0 && rloc < lp.N && col0 < lp.K) ptx::tma_store_2d(mC, sbuf, col0, rloc);
            if (lane == 0) ptx::bulk_commit();
            ++fchunk;
          }
        }
        if (fwd) lp.g_ring[((size_t)slot * 2 * lp.n_ct + (size_t)(c * 2 + hh)) * P.M + rloc + lane] = g;
      }
      // TMEM of this buffer is read: the MMA may refill it
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (even)
          ptx::mbar_arrive(&acce[buf]);
        else
          mbar_arrive_remote(&acce[buf], 0u);
      }
      // the task's outputs are written (TMA stores complete) before it is
      // counted done
      if (lane == 0) {
        bulk_wait_all();
        fence_proxy_async_global();
      }
      __threadfence();
      ptx::named_bar(BAR_EPI, 32 * EPI_WARPS);
      if (warp == EPI0 && lane == 0) {
        signal_done(P, task);
        if (even) trace_at(P, tidx, 5);
      }
    }
    if (lane == 0) bulk_wait_all();
  } else if (stream_cta) {
    // ----------------------------------------------------- streamers
    const int s = (int)threadIdx.x - 32 * STR0;
    int sidx = 0;
    for (int i = 0;; ++i) {
      uint2* slotp = stask_slot + (i & 1);
      if (s == 0) {
        const int idx = atomicAdd(P.cnt + C_QS, 1);
        uint2 t = idx < P.n_stask ? __ldg(P.stask + idx) : make_uint2(T_END, 0u);
        sidx = P.n_gtask + idx;
        if (t_type(t) != T_END) trace_at(P, sidx, 0);
        // the operands that do not wait on this batch start their way into
        // L2 now: an Adam chunk's W and moments, an overlay block's images
        if (t_type(t) == T_ADAM) {
          const LayerP& lp = P.lay[t_layer(t)];
          const int n0 = t_a(t) * ADAM_ROWS, n1 = n0 + ADAM_ROWS < lp.N ? n0 + ADAM_ROWS : lp.N;
          const size_t off = (size_t)n0 * lp.K, bytes = (size_t)(n1 - n0) * lp.K * 4;
          prefetch_l2(lp.W + off, bytes);
          prefetch_l2(lp.mW + off, bytes);
          prefetch_l2(lp.vW + off, bytes);
        } else if (t_type(t) == T_OV && P.xrp == 2 && (P.K0 & 3) == 0) {
          prefetch_l2(P.x + ((size_t)t_batch(t) * P.M + (size_t)t_a(t) * OV_ROWS) * P.K0, (size_t)OV_ROWS * P.K0 * 4);
        }
        if (t_type(t) != T_END && !wait_deps(P, t)) t = make_uint2(T_END, 0u);
        if (t_type(t) != T_END) trace_at(P, sidx, 1);
        *slotp = t;
      }
      ptx::named_bar(BAR_STR, NSTR);
      const uint2 t = *slotp;
      if (t_type(t) == T_END) break;
      switch (t_type(t)) {
        case T_OV: task_overlay(P, t_batch(t), t_a(t), s); break;
        case T_LG: task_local_grad(P, t_layer(t), t_batch(t), t_a(t), s, sred); break;
        case T_ADAM: task_adam(P, t_layer(t), t_batch(t), t_a(t), s); break;
      }
      __threadfence();
      ptx::named_bar(BAR_STR, NSTR);
      if (s == 0) {
        signal_done(P, t);
        trace_at(P, sidx, 5);
        trace_sm(P, sidx);
      }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::cluster_sync();
  ptx::tc_fence_after();
  if (warp == 1) ptx::tmem_dealloc_pair(tmem, TMEM_COLS);
}

}  // namespace

// ------------------------------------------------------------------- host
struct EpochPlan {
  int B = 0, nb = 0, xrp = 0;
  unsigned long long* trace = nullptr;  // [4 * (GEMM + stream tasks)] when tracing
  std::vector<void*> ws;   // each layer's workspace when the plan was built
  void* mem = nullptr;
  EpochP P{};
  int grid = 0;
  size_t counters_bytes = 0;
};

void epoch_plan_free(EpochPlan* p) {
  if (!p) return;
  dev_free(p->trace);
  dev_free(p->mem);
  delete p;
}

namespace {

size_t a256(size_t b) { return (b + 255) & ~(size_t)255; }

// Builds the task tables, rings, tensor maps and counters of an epoch of nb
// full batches of B pairs through the net's layers.
ff_status build_plan(ff_net* n, int B, int nb, int xrp, cudaStream_t st, EpochPlan** out) {
  const int L = n->L, D = n->depth < 2 ? 2 : (n->depth > kMaxSlots ? kMaxSlots : n->depth), M = 2 * B;
  std::vector<ff_layer*>& Ls = n->layers;
  // task tables, in the global order: per tick, FWD tiles, then the stream
  // queue's overlay of the next batch and local gradients, then WG tiles,
  // then Adam chunks
  std::vector<uint2> gt, stt;
  const int rts = M / BN;
  for (int r = 0; r < M / OV_ROWS; ++r) stt.push_back(mk_task(T_OV, 0, 0, r, 0));
  const int ticks = nb + L - 1;
  for (int tau = 0; tau < ticks; ++tau) {
    for (int k = 0; k < L; ++k) {
      const int b = tau - k;
      if (b < 0 || b >= nb) continue;
      const int nct = cdiv(Ls[k]->N, BN);
      for (int rt = 0; rt < rts; ++rt)
        for (int ct = 0; ct < nct; ++ct) gt.push_back(mk_task(T_FWD, k, b, rt, ct));
    }
    if (tau + 1 < nb)
      for (int r = 0; r < M / OV_ROWS; ++r) stt.push_back(mk_task(T_OV, 0, tau + 1, r, 0));
    for (int k = 0; k < L; ++k) {
      const int b = tau - k;
      if (b < 0 || b >= nb) continue;
      for (int rb = 0; rb < M / LG_TASK_ROWS; ++rb) stt.push_back(mk_task(T_LG, k, b, rb, 0));
    }
    for (int k = 0; k < L; ++k) {
      const int b = tau - k;
      if (b < 0 || b >= nb) continue;
      const int nnt = cdiv(Ls[k]->N, BN), nkt = cdiv(Ls[k]->K, BN);
      for (int nt = 0; nt < nnt; ++nt)
        for (int kt = 0; kt < nkt; ++kt) gt.push_back(mk_task(T_WG, k, b, nt, kt));
    }
    for (int k = 0; k < L; ++k) {
      const int b = tau - k;
      if (b < 0 || b >= nb) continue;
      for (int c = 0; c < cdiv(Ls[k]->N, ADAM_ROWS); ++c) stt.push_back(mk_task(T_ADAM, k, b, c, 0));
    }
  }
  // device memory: counters, tasks, maps, rings
  size_t off = 0;
  const size_t oCnt = off; off += a256((size_t)N_COUNTERS * 4);
  const size_t oGT = off; off += a256(gt.size() * sizeof(uint2));
  const size_t oST = off; off += a256(stt.size() * sizeof(uint2));
  const size_t oTM = off; off += a256((size_t)L * TM_N * sizeof(CUtensorMap));
  const int ldK0 = Ls[0]->ldK;
  const size_t oX0 = off; off += a256((size_t)D * M * ldK0 * 2);
  const size_t oS0 = off; off += a256((size_t)D * M * 4);
  std::vector<size_t> oH(L), oG(L), oSN(L);
  for (int k = 0; k < L; ++k) {
    oH[k] = off; off += a256((size_t)D * M * Ls[k]->ldN * 2);
    oG[k] = off; off += a256((size_t)D * 2 * cdiv(Ls[k]->N, BN) * M * 4);
    oSN[k] = off; off += a256(k + 1 < L ? (size_t)D * M * 4 : 0);
  }
  EpochPlan* p = new (std::nothrow) EpochPlan();
  if (!p) return FF_ERR_OOM;
  ff_status s = cuda_status(dev_alloc(&p->mem, off), "epoch plan memory");
  if (s != FF_OK) {
    delete p;
    return s;
  }
  char* base = static_cast<char*>(p->mem);
  EpochP& P = p->P;
  P.L = L;
  P.D = D;
  P.M = M;
  P.B = B;
  P.nb = nb;
  P.xrp = xrp;
  P.K0 = Ls[0]->K;
  P.ldK0 = ldK0;
  P.x0_ring = reinterpret_cast<bf16*>(base + oX0);
  P.s0_ring = reinterpret_cast<float*>(base + oS0);
  P.gtask = reinterpret_cast<const uint2*>(base + oGT);
  P.n_gtask = (int)gt.size();
  P.stask = reinterpret_cast<const uint2*>(base + oST);
  P.n_stask = (int)stt.size();
  P.cnt = reinterpret_cast<int*>(base + oCnt);
  P.err = &Ls[0]->ds->err;
  std::vector<CUtensorMap> maps((size_t)L * TM_N);
  bool maps_ok = true;
  for (int k = 0; k < L; ++k) {
    ff_layer* Lk = Ls[k];
    LayerP& lp = P.lay[k];
    lp.K = Lk->K;
    lp.N = Lk->N;
    lp.ldK = Lk->ldK;
    lp.ldN = Lk->ldN;
    lp.n_ct = cdiv(Lk->N, BN);
    lp.n_kt = cdiv(Lk->K, BN);
    lp.n_chunks = cdiv(Lk->N, ADAM_ROWS);
    lp.has_bias = Lk->cfg.has_bias;
    lp.discard_dW = !Lk->cfg.keep_grad && ((uintptr_t)Lk->dW & 127u) == 0;
    lp.theta = Lk->cfg.theta;
    lp.lr = Lk->cfg.lr;
    lp.beta1 = Lk->cfg.beta1;
    lp.beta2 = Lk->cfg.beta2;
    lp.eps = Lk->cfg.eps;
    lp.beta1d = Lk->cfg.beta1;
    lp.beta2d = Lk->cfg.beta2;
    const bf16* in_ring = k == 0 ? P.x0_ring : reinterpret_cast<const bf16*>(base + oH[k - 1]);
    lp.s_in_ring = k == 0 ? P.s0_ring : reinterpret_cast<const float*>(base + oSN[k - 1]);
    lp.h_ring = reinterpret_cast<bf16*>(base + oH[k]);
    lp.g_ring = reinterpret_cast<float*>(base + oG[k]);
    lp.sn_ring = k + 1 < L ? reinterpret_cast<float*>(base + oSN[k]) : nullptr;
    lp.dZ = static_cast<bf16*>(Lk->dZ);
    lp.dW = Lk->dW;
    lp.W = Lk->W;
    lp.mW = Lk->mW;
    lp.vW = Lk->vW;
    lp.b = Lk->b;
    lp.mb = Lk->mb;
    lp.vb = Lk->vb;
    lp.db_out = Lk->db;
    lp.Wb = Lk->Wb;
    lp.dbpart = Lk->dbpart;
    lp.loss_part = Lk->loss_part;
    lp.stat_part = Lk->stat_part;
    lp.ds = Lk->ds;
    lp.tm = reinterpret_cast<const CUtensorMap*>(base + oTM) + (size_t)k * TM_N;
    CUtensorMap* m = &maps[(size_t)k * TM_N];
    maps_ok = maps_ok && make_sw128_map(&m[TM_FWD_A], in_ring, 2, Lk->K, D * M, Lk->ldK, BK, BM) &&
              make_sw128_map(&m[TM_FWD_B], Lk->Wb, 2, Lk->K, Lk->N, Lk->ldK, BK, HB) &&
              make_sw128_map(&m[TM_FWD_C], lp.h_ring, 2, Lk->ldN, D * M, Lk->ldN, 64, 32) &&
              make_sw128_map(&m[TM_WG_A], Lk->dZ, 2, Lk->N, M, Lk->ldN, 64, BK) &&
              make_sw128_map(&m[TM_WG_B], in_ring, 2, Lk->K, D * M, Lk->ldK, 64, BK) &&
              make_sw128_map(&m[TM_WG_C], Lk->dW, 4, Lk->K, Lk->N, Lk->K, 32, 32);
  }
  if (!maps_ok) {
    epoch_plan_free(p);
    return FF_ERR_INVALID_ARG;
  }
  s = cuda_status(cudaMemcpyAsync(base + oGT, gt.data(), gt.size() * sizeof(uint2), cudaMemcpyHostToDevice, st),
                  "epoch task table");
  if (s == FF_OK)
    s = cuda_status(cudaMemcpyAsync(base + oST, stt.data(), stt.size() * sizeof(uint2), cudaMemcpyHostToDevice, st),
                    "epoch task table");
  if (s == FF_OK)
    s = cuda_status(cudaMemcpyAsync(base + oTM, maps.data(), maps.size() * sizeof(CUtensorMap),
                                    cudaMemcpyHostToDevice, st),
                    "epoch tensor maps");
  if (s == FF_OK) s = cuda_status(cudaStreamSynchronize(st), "epoch plan upload");
  if (s != FF_OK) {
    epoch_plan_free(p);
    return s;
  }
  static cudaError_t attr = cudaFuncSetAttribute(k_epoch, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (attr != cudaSuccess) {
    epoch_plan_free(p);
    return cuda_status(attr, "epoch kernel attributes");
  }
  // one CTA per SM, in pairs: as many pairs as can be resident at once
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(NTHREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int clusters = 0;
  s = cuda_status(cudaOccupancyMaxActiveClusters(&clusters, k_epoch, &cfg), "epoch occupancy");
  if (std::getenv("FF_DEBUG")) {
    cudaFuncAttributes fa{};
    cudaFuncGetAttributes(&fa, k_epoch);
    int per_sm = -1;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_epoch, NTHREADS, SMEM_BYTES);
    std::fprintf(stderr,
                 "[ff] epoch kernel: regs %d, max threads %d, static smem %zu, dynamic smem %d (max %d), "
                 "blocks/SM %d, clusters %d, status %d\n",
                 fa.numRegs, fa.maxThreadsPerBlock, fa.sharedSizeBytes, SMEM_BYTES, fa.maxDynamicSharedSizeBytes,
                 per_sm, clusters, (int)s);
  }
  if (s != FF_OK || clusters < 1) {
    epoch_plan_free(p);
    return s != FF_OK ? s : FF_ERR_UNSUPPORTED;
  }
  p->grid = 2 * clusters;
  p->P.gemm_clusters = clusters;
  p->P.split = 0;
  if (const char* g = std::getenv("FF_EPOCH_GEMM_CLUSTERS")) {
    // split the roles: this many clusters run GEMM tiles only, the rest stream
    const int gc = std::atoi(g);
    if (gc >= 1 && gc < clusters) {
      p->P.gemm_clusters = gc;
      p->P.split = 1;
    }
  }
  for (int k = 0; k < L; ++k) p->ws.push_back(Ls[k]->X);
  p->B = B;
  p->nb = nb;
  p->xrp = xrp;
  p->counters_bytes = (size_t)N_COUNTERS * 4;
  *out = p;
  return FF_OK;
}

}  // namespace

ff_status net_train_epoch(ff_net* n, const float* x, const int* labels, int n_pairs, int B, int xrp, float* loss,
                          cudaStream_t st) {
  const int L = n->L;
  const int nb = n_pairs / B, tail = n_pairs % B;
  for (int k = 0; k < L; ++k) {
    ff_status s = ensure_capacity(n->layers[k], 2 * B);
    if (s != FF_OK) return s;
  }
  // the layer streams' earlier work comes first
  for (int k = 0; k < L; ++k) {
    cudaError_t e = cudaEventRecord(n->tail[k], n->streams[k]);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, n->tail[k], 0);
    FF_TRY(e, "epoch: join layer streams");
  }
  if (nb > 0) {
    EpochPlan* p = n->epoch;
    bool stale = !p || p->B != B || p->nb != nb || p->xrp != xrp;
    for (int k = 0; k < L && !stale; ++k) stale = p->ws[k] != n->layers[k]->X;
    if (stale) {
      FF_TRY(cudaStreamSynchronize(st), "epoch: sync before re-planning");
      epoch_plan_free(p);
      n->epoch = nullptr;
      ff_status s = build_plan(n, B, nb, xrp, st, &n->epoch);
      if (s != FF_OK) return s;
      p = n->epoch;
    }
    EpochP P = p->P;
    if (n->epoch_trace && !p->trace) {
      const size_t bytes = (size_t)kTraceWords * (p->P.n_gtask + p->P.n_stask) * sizeof(unsigned long long);
      FF_TRY(dev_alloc(reinterpret_cast<void**>(&p->trace), bytes), "epoch trace");
      FF_TRY(cudaMemsetAsync(p->trace, 0, bytes, st), "epoch trace");
    }
    P.trace = n->epoch_trace ? p->trace : nullptr;
    P.x = x;
    P.labels = labels;
    P.loss = loss;
    FF_TRY(cudaMemsetAsync(P.cnt, 0, p->counters_bytes, st), "epoch counters");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p->grid, 1, 1);
    cfg.blockDim = dim3(NTHREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    double flops = 0;
    for (int k = 0; k < L; ++k) flops += 4.0 * (2.0 * B) * n->layers[k]->N * n->layers[k]->K;
    FF_LAUNCH(K_EPOCH, flops * nb, st, cudaLaunchKernelEx(&cfg, k_epoch, P), "persistent train epoch");
    for (int k = 0; k < L; ++k) n->layers[k]->last_stream = st;
  }
  n->since_sync = 0;
  if (tail > 0) {
    const float* xt = x + (size_t)nb * (size_t)B * (size_t)xrp * (size_t)n->layers[0]->K;
    ff_status s = net_train_step(n, xt, labels + (size_t)nb * 2 * B, tail, loss ? loss + (size_t)nb * L : nullptr,
                                 st, xrp == 1);
    if (s != FF_OK) return s;
  }
  return ff_net_sync(n, st);
}

}  // namespace ff

extern "C" FF_API ff_status ff_net_train_epoch(ff_net* n, const float* x, const int* labels, int n_pairs, int B,
                                               int images_per_pair_row, float* loss, void* stream) {
  ff::NvtxRange nvtx_("ff_net_train_epoch");
  if (!n || !x || !labels || n_pairs < 0 || B < 1 || B > n->max_B || n->po) return FF_ERR_INVALID_ARG;
  if (images_per_pair_row != 1 && images_per_pair_row != 2) return FF_ERR_INVALID_ARG;
  if (n_pairs == 0) return FF_OK;
  if ((reinterpret_cast<uintptr_t>(x) & 3u) != 0) return FF_ERR_INVALID_ARG;
  const int L = n->L;
  bool persistent = L <= ff::kMaxLayers && (2 * B) % ff::BN == 0 && (2 * B) / ff::BN <= ff::kMaxTiles &&
                    ff::tc_supported();
  for (int k = 0; k < L && persistent; ++k) {
    const ff_layer* l = n->layers[k];
    persistent = l->is_bf16 && l->K % 8 == 0 && l->N % 8 == 0 && ff::cdiv(l->N, ff::BN) <= ff::kMaxTiles &&
                 l->N <= 65535 && l->K <= 65535;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (!persistent) {
    // the same batches one step at a time on the layer streams
    for (int done = 0, t = 0; done < n_pairs; ++t) {
      const int b = n_pairs - done < B ? n_pairs - done : B;
      const float* xb = x + (size_t)done * images_per_pair_row * n->layers[0]->K;
      ff_status s = ff::net_train_step(n, xb, labels + (size_t)2 * done, b, loss ? loss + (size_t)t * L : nullptr,
                                       stream, images_per_pair_row == 1);
      if (s != FF_OK) return s;
      done += b;
    }
    return ff_net_sync(n, stream);
  }
  return ff::net_train_epoch(n, x, labels, n_pairs, B, images_per_pair_row, loss, st);
}

extern "C" FF_API long long ff_net_epoch_trace(ff_net* n, int enable, unsigned long long* out, long long capacity) {
  if (!n) return -1;
  if (enable >= 0) n->epoch_trace = enable != 0;
  if (!out) return 0;
  ff::EpochPlan* p = n->epoch;
  if (!p || !p->trace || capacity < 2) return 0;
  const long long recs = (long long)p->P.n_gtask + p->P.n_stask;
  long long words = ff::kTraceWords * recs;
  if (words > capacity - 2) words = (capacity - 2) / ff::kTraceWords * ff::kTraceWords;
  if (cudaDeviceSynchronize() != cudaSuccess) return -1;
  out[0] = (unsigned long long)p->P.n_gtask;
  out[1] = (unsigned long long)p->P.n_stask;
  if (cudaMemcpy(out + 2, p->trace, (size_t)words * sizeof(unsigned long long), cudaMemcpyDeviceToHost) != cudaSuccess)
    return -1;
  return words + 2;
}
