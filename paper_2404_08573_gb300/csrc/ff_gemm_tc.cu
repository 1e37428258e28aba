// Tensor-core GEMMs of the FF layer step (bf16 operands, fp32 accumulate in
// TMEM), written for sm_103a with tcgen05 + TMA:
//
//   forward  Z = diag(s) X W^T + b, H = ReLU(Z), per-tile goodness partials
//            (the linear+ReLU of §3 on the concatenated batch of §4, and the
//            sum of squared activities of Eq. 1 taken from the fp32
//            accumulator);
//            -- optionally also per-tile partial logits of a 10-class
//            softmax block on the stored activity (the Performance-
//            Optimized layer of §4);
//   store    C = X W^T in fp32 (the label-free part of layer 1 in predict);
//   wgrad    dW = G^T X with G = diag(s) dZ, contracting over the batch rows
//            (both operands are read MN-major straight from their row-major
//            buffers: no transposed copies);
//   forward with the local gradient (train step): the forward above, and in
//            the same epilogue the rest of the layer's local step of §3
//            (Eq. 1): each row's goodness summed over all column tiles, the
//            loss, dL/dg, the next layer's row scale, the weight-gradient
//            operand dZ' = s * 2 dL/dg * h and the bias-gradient partials.
//            The CTAs holding a row block's column tiles form one cluster and
//            exchange their goodness partials through distributed shared
//            memory (plain remote stores and remote mbarrier arrivals).
//
// One CTA computes one (MT*BM) x (NT*BN) output tile with three warp roles:
//   warp 0      TMA producer: 128-byte-swizzled tiles into a STAGES-deep ring
//   warp 1      allocates TMEM, one elected lane issues tcgen05.mma (M=128,
//               N=BN, K=16; one per row subtile and column subtile, each
//               into its own accumulator) and commits each stage back to the
//               producer
// In pair mode two CTAs (a cluster of 2 along x) run as one cta_group::2
// unit: each loads its own A rows and half of B, the even CTA's MMA warp
// issues M=256 MMAs over both, and each CTA's epilogue reads its own TMEM.
//   warps 2..9  epilogue: tcgen05.ld of TMEM lanes 32*(warp%4).., one half of
//               the columns each -> registers, fused scale/bias/ReLU/goodness
//               (partials per 128-column half) or plain store
// fp32 operands (OPB = 4, the exact-precision mode's forward and store
// GEMMs): the tensor cores' TF32 products in three terms, A B ~ Ah Bh + Ah Bl +
// Al Bh, where xh is x with the 13 low mantissa bits cleared (exactly a TF32
// value) and xl = x - xh (exact in fp32); the dropped Al Bl and the TF32
// truncation of xl leave a relative error near 2^-21 per product.  The
// epilogue warps, idle during the mainloop, split each landed stage in
// shared memory (hi in place, lo beside it) before the MMAs read it.
// Every mbarrier wait is bounded (kWaitTimeoutNs); a timeout latches
// DEVERR_TIMEOUT in *err, tells the other roles to stop, waits for copies and
// MMAs already in flight and frees TMEM before the CTA exits.
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstdlib>
#include <mutex>

#include "ff_internal.cuh"
#include "ff_ptx.cuh"

namespace ff {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // one 128-byte swizzle row of bf16
constexpr int EPI_WARPS = 8;                 // two per TMEM lane quarter, each on half the columns
constexpr int NTHREADS = 64 + 32 * EPI_WARPS;  // producer warp, MMA warp, epilogue warps
constexpr int MODE_FWD = 0;
constexpr int MODE_STORE = 1;
constexpr int MODE_FWD_LOGITS = 2;  // forward, plus partial logits of a 10-class block (EpiArgs::logit_V)
constexpr int MODE_FWD_LG = 3;      // forward, plus the local gradient (GradPrepArgs), cluster-wide goodness
constexpr int kLgParts = 16;        // goodness partials of a row (128 columns each) a cluster can hold
constexpr int kLogitClasses = 10;
constexpr int kLogitStride = 12;    // floats per column of the staged block weights (three float4)

template <int BN, int NSTAGE, int MT, bool PAIR, int NT = 1, int OPB = 2, int KB = 128>
struct TcCfg {
  // OPB: bytes per operand element (2: bf16; 4: fp32 through three TF32
  // products).  KB: bytes of K per operand row of a stage -- one 128-byte
  // swizzle row, or (bf16 only) one 64-byte swizzle row, which halves the
  // stage so that twice as many fit the same ring.  A stage holds BKE = KB /
  // OPB elements of K, so tile byte sizes do not depend on the type.
  static constexpr int KBYTES = KB;
  static constexpr int BKE = KB / OPB;
  static constexpr int TN = NT * BN;                // columns of the tile (NT column subtiles of BN)
  static constexpr int A_BYTES = MT * BM * KB;      // MT row subtiles of BM rows
  static constexpr int BH = PAIR ? BN / 2 : BN;     // B columns of a column subtile this CTA loads
  static constexpr int B_BYTES = NT * BH * KB;
  static constexpr int IN_BYTES = A_BYTES + B_BYTES;  // what TMA brings per stage
  static constexpr int STAGE = (OPB == 4 ? 2 : 1) * IN_BYTES;  // fp32: the lo parts beside
  static constexpr int STAGES = NSTAGE;
  static constexpr int SMEM = STAGES * STAGE + 1024 /*alignment slack*/ + 256 /*barriers*/ + TN * 4 /*bias*/;
  // the local-gradient epilogue: every partial of the cluster's row block,
  // and per epilogue warp its rows' 2 dL/dg and s 2 dL/dg
  static constexpr int LG_SMEM = kLgParts * MT * BM * 4 + EPI_WARPS * 32 * 2 * 4;
  static constexpr uint32_t ACC_COLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  static constexpr uint32_t TMEM_COLS = MT * NT * ACC_COLS;  // one accumulator per (row, column) subtile
  static_assert(BN % 64 == 0 && BN <= 256, "BN must be a multiple of 64, at most 256");
  static_assert(MT >= 1 && NT >= 1 && MT * NT * ACC_COLS <= 512, "accumulators must fit in TMEM");
  static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
  static_assert(OPB == 4 || MT * 4 * 32 * TN * 2 <= STAGES * STAGE, "bf16 epilogue staging must fit in the operand ring");
  static_assert(OPB == 2 || OPB == 4, "bf16 or fp32 operands");
  static_assert(KB == 128 || (KB == 64 && OPB == 2), "128-byte K rows, or 64-byte ones for bf16");
  static_assert(EPI_WARPS * 8192 <= STAGES * STAGE, "fp32 epilogue staging must fit in the operand ring");
  static_assert(TN % (64 * (EPI_WARPS / 4)) == 0, "each epilogue warp takes whole 64-column groups");
  static_assert(NT == 1 || TN / (EPI_WARPS / 4) == BN, "with column subtiles each epilogue warp reads one accumulator");
  static_assert(!PAIR || BH % 64 == 0, "each CTA of a pair loads whole 64-column B groups");
  static_assert(3 * STAGES * 8 + 8 + 16 + 8 + 32 <= 256, "barriers, TMEM slot, flags, LG and logits barriers fit below the bias");
};

__device__ __forceinline__ void latch(int* err, volatile int* abort_flag) {
  *abort_flag = 1;
  atomicOr(err, DEVERR_TIMEOUT);
}

// The kernel: one body (ff_gemm_tc_body.inc) compiled into two kernels that
// differ only in their register bound.
//   k_tc_gemm: at most 96 registers a thread (the bound for two CTAs of 320
//   threads per SM; no spills), so a CTA leaves room on its SM for the Adam
//   and local-gradient blocks of the other layers' streams (784-2000x4 epoch
//   -1 %).
//   k_tc_gemm_r88: at most 88, for the instances with 64-byte K rows (the
//   two-subtile train-step GEMMs): an SM then fits three 256-thread Adam
//   blocks of 48 registers beside the GEMM CTA instead of two (784-2000x4
//   epoch 7.82 -> 7.73 ms; at 80 registers the forward's epilogue spills and
//   the gain is gone).  A launch bound cannot ask for 88 (it divides the
//   registers by whole warps per SM sub-partition), hence __maxnreg__.
// MODE_FWD_LG: tmD maps dZ' (as tmC maps H) and lg holds the local step's
// arguments; the grid's column tiles all lie in one cluster (2 x gridDim.y).
template <int BN, bool A_MN, bool B_MN, int MODE, bool PAIR, int NSTAGE, int MT, int NT, int OPB, int KB>
__global__ void __launch_bounds__(NTHREADS, 2)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmD, int tma_store, int M,
              int N, int K, EpiArgs ep, GradPrepArgs lg, int* err) {
#include "ff_gemm_tc_body.inc"
}

template <int BN, bool A_MN, bool B_MN, int MODE, bool PAIR, int NSTAGE, int MT, int NT, int OPB, int KB>
__global__ void __maxnreg__(88)
    k_tc_gemm_r88(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmD, int tma_store,
                  int M, int N, int K, EpiArgs ep, GradPrepArgs lg, int* err) {
#include "ff_gemm_tc_body.inc"
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Row-major matrix [rows, cols] of bf16 (esize 2) or fp32 (esize 4) with row
// stride ld (elements), tiled in boxes of box_rows x box_cols with 128-byte
// swizzle; out-of-range elements of a box read as zero and are not written.
bool encode_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols, int box_rows,
                CUtensorMapSwizzle swz) {
  auto enc = encode_fn();
  if (!enc) return false;
  if ((reinterpret_cast<uintptr_t>(ptr) & 15u) || ((size_t)ld * esize) % 16 != 0) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)ld * esize};
  cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, esize == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
             const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
bool make_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols, int box_rows) {
  return encode_map(m, ptr, esize, cols, rows, ld, box_cols, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}
// A K-major bf16 operand [rows, K] in boxes of box_rows rows and one stage's
// K row of kb bytes (128: 128-byte swizzle; 64: 64-byte swizzle).
bool make_kmajor_map(CUtensorMap* m, const bf16* ptr, int K, int rows, int ld, int box_rows, int kb) {
  return encode_map(m, ptr, 2, K, rows, ld, kb / 2, box_rows,
                    kb == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B);
}

template <int BN, int NSTAGE, int MT, bool PAIR, int NT, int MODE, int OPB, int KB>
constexpr int tc_smem() {
  using C = TcCfg<BN, NSTAGE, MT, PAIR, NT, OPB, KB>;
  return C::SMEM + (MODE == MODE_FWD_LOGITS ? BN * kLogitStride * 4 : 0) + (MODE == MODE_FWD_LG ? C::LG_SMEM : 0);
}

// Launch configuration of one instance: the grid (tile rows padded to whole
// pairs; a padding CTA loads zeros, supplies its half of B and writes
// nothing), clusters of the pair (LG: of the pair and every column tile),
// and programmatic stream serialization.
template <int BN, bool A_MN, bool B_MN, int MODE, bool PAIR, int NSTAGE, int MT, int NT, int OPB = 2, int KB = 128>
struct TcLaunch {
  static constexpr int SMEM = tc_smem<BN, NSTAGE, MT, PAIR, NT, MODE, OPB, KB>();
  static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
  // More than half of an SM's 228 KB (with the 1 KB each CTA reserves): no
  // two GEMM CTAs, of this or any other instance, share an SM, so no TMEM
  // allocation waits for another CTA's (a pair waiting on a pair could
  // otherwise deadlock).
  static_assert(SMEM > 113 * 1024, "a GEMM CTA must hold more than half of its SM's shared memory");
  static constexpr int CM = PAIR ? 2 : 1;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[2];
  TcLaunch(int M, int N, cudaStream_t st) {
    cfg.gridDim = dim3(cdiv(cdiv(M, BM * MT), CM) * CM, cdiv(N, NT * BN), 1);
    cfg.blockDim = dim3(NTHREADS, 1, 1);
    cfg.dynamicSmemBytes = SMEM;
    cfg.stream = st;
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = CM;
    at[0].val.clusterDim.y = MODE == MODE_FWD_LG ? cfg.gridDim.y : 1;
    at[0].val.clusterDim.z = 1;
    // the next kernel's launch and set-up overlap this one's tail (griddep_*)
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
  }
  static auto kernel() {
    if constexpr (KB == 64)
      return k_tc_gemm_r88<BN, A_MN, B_MN, MODE, PAIR, NSTAGE, MT, NT, OPB, KB>;
    else
      return k_tc_gemm<BN, A_MN, B_MN, MODE, PAIR, NSTAGE, MT, NT, OPB, KB>;
  }
  static cudaError_t set_attrs() {
    static cudaError_t e = cudaFuncSetAttribute(kernel(), cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    return e;
  }
};

template <int BN, bool A_MN, bool B_MN, int MODE, bool PAIR, int NSTAGE, int MT, int NT = 1, int OPB = 2,
          int KB = 128>
cudaError_t launch_tc(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc, int tma_store, int M, int N,
                      int K, const EpiArgs& ep, int* err, cudaStream_t st, const CUtensorMap* td = nullptr,
                      const GradPrepArgs* lg = nullptr) {
  using Lc = TcLaunch<BN, A_MN, B_MN, MODE, PAIR, NSTAGE, MT, NT, OPB, KB>;
  const cudaError_t attr = Lc::set_attrs();
  if (attr != cudaSuccess) return attr;
  Lc l(M, N, st);
  const GradPrepArgs none{};
  return cudaLaunchKernelEx(&l.cfg, Lc::kernel(), ta, tb, tc, td ? *td : tc, tma_store, M, N, K, ep, lg ? *lg : none,
                            err);
}

constexpr int FWD_BN = 256;
constexpr int WGRAD_BN = 256;
// Tile configuration: CTA pairs (cta_group::2) with two 128-row subtiles per
// CTA, so a pair computes a 512 x 256 tile; per 64-deep K step a CTA loads
// 48 KB of operands (its 256 A rows, half of B) for 8.4 MFLOP.  Measured on
// the 784-2000x4 train step with the layers on 4 streams (epoch, ms):
//   single CTA 256 x 256 (two subtiles), 3-stage ring ........... 9.30
//   pairs, one subtile per CTA (128 CTAs per GEMM), 6 / 4 stages  9.90 / 10.52
//   pairs, two subtiles per CTA (64 CTAs per GEMM), 4 / 3 stages  9.05 / 8.78
// With 128 CTAs a GEMM alone is faster (20 vs 29 us for 2048x2000x2000) but
// two layers' GEMMs no longer fit on the GPU side by side (re-measured with
// dependent launch and the later Adam changes: 9.54 against 8.32 ms); earlier
// 128 x 256 tiles and 4-CTA multicast clusters measured 9.8 and 11.1 ms.
// The ring of the two-subtile forward, store and weight-gradient GEMMs holds
// 144 KB either as 3 stages of 64-deep K steps (128-byte rows) or as 6
// stages of 32-deep ones (64-byte rows, 24 KB).  The finer ring keeps 120 KB
// of operand loads in flight instead of 96 KB: an epoch's forward GEMMs, one
// at a time, 6.61 -> 6.10-6.19 ms; the epoch 8.10 -> 7.95 ms.  Deeper rings of 24 KB
// stages are faster alone but slower in the epoch, as the 4-stage ring of
// 48 KB was (7 / 8 stages: 8.00 / 8.57 ms): past ~170 KB a GEMM CTA leaves
// too little of its SM to the other streams' blocks.
constexpr bool USE_PAIR = true;
constexpr int NSTAGES = 3;       // operand ring depth with 128-byte K rows (48 KB stages)
constexpr int ROW_SUBTILES = 2;  // 128-row subtiles per CTA (each with its own TMEM accumulator)
constexpr int KB_FULL = 64;      // bytes of K per operand row of a stage, two-subtile GEMMs
constexpr int NSTAGES_FULL = 6;  // their ring depth
constexpr int CLUSTER_M = USE_PAIR ? 2 : 1;
// A GEMM that would get fewer than kSmallGridCtas CTAs with two subtiles per
// CTA (at most a third of the GPU, e.g. 1216 batch rows of a 2000-wide
// layer) runs with one subtile per CTA instead: twice the CTAs, each with a
// 4-stage ring of 32 KB stages (128-byte rows).  One whose one-subtile grid
// still fills at most half the SMs (1024 rows of a 2000-wide layer: 64 CTAs)
// also halves the tile width to 128 columns (128 CTAs, 8-stage ring of 24 KB
// stages).  The one-subtile ring, on the epoch (layer 1's weight gradient):
// 6 / 5 / 4 stages of 32 KB 7.90 / 7.89 / 7.81 ms -- the smaller footprint
// again leaves more of the SM to the other streams; 8 stages of 16 KB
// (64-byte rows, 128 KB) 7.98 ms.  Every ring keeps a CTA above half an
// SM's shared memory, so two GEMM CTAs, whose TMEM allocations could then
// wait on each other, never share an SM.
constexpr int kSmallGridCtas = 64;
constexpr int NSTAGES_SMALL = 4;
constexpr int TINY_BN = 128;
constexpr int kTinyGridCtas = 152 / 2;
constexpr int NSTAGES_TINY = 8;
enum Shape { SHAPE_FULL, SHAPE_SMALL, SHAPE_TINY };
int grid_ctas(int M, int N, int mt, int bn) { return cdiv(cdiv(M, BM * mt), CLUSTER_M) * CLUSTER_M * cdiv(N, bn); }
Shape shape_of(int M, int N, int bn) {
  if (grid_ctas(M, N, ROW_SUBTILES, bn) >= kSmallGridCtas) return SHAPE_FULL;
  return grid_ctas(M, N, 1, bn) > kTinyGridCtas ? SHAPE_SMALL : SHAPE_TINY;
}

}  // namespace

bool make_plain_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols,
                    int box_rows) {
  return encode_map(m, ptr, esize, cols, rows, ld, box_cols, box_rows, CU_TENSOR_MAP_SWIZZLE_NONE);
}

bool make_sw128_map(CUtensorMap* m, const void* ptr, int esize, int cols, int rows, int ld, int box_cols,
                    int box_rows) {
  return make_map(m, ptr, esize, cols, rows, ld, box_cols, box_rows);
}

bool tc_supported() {
  int dev = 0, major = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
  return major == 10 && encode_fn() != nullptr;
}

// goodness partials per row: one per epilogue warp's column half of each column tile
int tc_fwd_ntiles(int M, int N, bool narrow) {
  return cdiv(N, narrow && shape_of(M, N, FWD_BN) == SHAPE_TINY ? TINY_BN : FWD_BN) * (EPI_WARPS / 4);
}
int tc_fwd_ntiles_max(int N) { return cdiv(N, TINY_BN) * (EPI_WARPS / 4); }

int tc_gemm_fwd_ctas(int M, int N, bool narrow) {
  switch (shape_of(M, N, FWD_BN)) {
    case SHAPE_FULL: return grid_ctas(M, N, ROW_SUBTILES, FWD_BN);
    case SHAPE_SMALL: return grid_ctas(M, N, 1, FWD_BN);
    default: return grid_ctas(M, N, 1, narrow ? TINY_BN : FWD_BN);
  }
}

// B (the weights, [N, K]) is loaded per CTA in boxes of the CTA's share of a tile's columns.
static constexpr int b_box_rows(int bn) { return USE_PAIR ? bn / 2 : bn; }

// The train step's forward with the local gradient: CTA pairs of 256 rows x
// 512 columns (two 256-column accumulators per CTA; per 64-deep K step a CTA
// loads 48 KB of operands for 8.4 MFLOP, as the 512 x 256 pairs above) and
// every column tile of a row block in one cluster, so at most 4 column tiles
// (N <= 2048) in the portable cluster size of 8.
using FwdLg = TcLaunch<FWD_BN, false, false, MODE_FWD_LG, true, NSTAGES, 1, 2>;
constexpr int kLgMaxColTiles = 4;

bool tc_fwd_lg_supported(int M, int N) {
  if (M <= 0 || N <= 0 || cdiv(N, 2 * FWD_BN) > kLgMaxColTiles) return false;
  // clusters of 2 x (column tiles) CTAs must fit the GPU (checked once per column-tile count)
  static int ok[kLgMaxColTiles + 1] = {0, 0, 0, 0, 0};  // 0 unknown, 1 yes, -1 no
  const int ct = cdiv(N, 2 * FWD_BN);
  if (ok[ct] == 0) {
    int clusters = 0;
    cudaError_t e = FwdLg::set_attrs();
    if (e == cudaSuccess) {
      // the occupancy query takes the cluster shape alone (no other launch attributes)
      FwdLg l(2 * BM, ct * 2 * FWD_BN, nullptr);
      l.cfg.numAttrs = 1;
      e = cudaOccupancyMaxActiveClusters(&clusters, FwdLg::kernel(), &l.cfg);
    }
    if (e != cudaSuccess) cudaGetLastError();  // leave no sticky launch-configuration error behind
    if (std::getenv("FF_DEBUG"))
      std::fprintf(stderr, "[ff] forward with local gradient, %d column tiles: %d clusters of %d CTAs (%s)\n", ct,
                   clusters, 2 * ct, cudaGetErrorString(e));
    ok[ct] = e == cudaSuccess && clusters > 0 ? 1 : -1;
  }
  return ok[ct] > 0;
}

cudaError_t tc_gemm_fwd_lg(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                           const GradPrepArgs& lg, bf16* dZ, int* err, cudaStream_t st) {
  if (!tc_fwd_lg_supported(M, N) || ep.gpart_in || ep.logit_V || !lg.loss_part || !lg.dbpart)
    return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tc, td;
  if (!make_map(&ta, A, 2, K, M, lda, BK, BM) || !make_map(&tb, B, 2, K, N, ldb, BK, b_box_rows(FWD_BN)) ||
      !make_map(&tc, ep.out, 2, ep.ldo, M, ep.ldo, 64, 32) || !make_map(&td, dZ, 2, ep.ldo, M, ep.ldo, 64, 32))
    return cudaErrorInvalidValue;
  return launch_tc<FWD_BN, false, false, MODE_FWD_LG, true, NSTAGES, 1, 2>(ta, tb, tc, 1, M, N, K, ep, err, st, &td,
                                                                            &lg);
}

cudaError_t tc_gemm_fwd(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                        int* err, cudaStream_t st) {
  Shape sh = shape_of(M, N, FWD_BN);
  if (sh == SHAPE_TINY && !ep.narrow) sh = SHAPE_SMALL;
  const int bn = sh == SHAPE_TINY ? TINY_BN : FWD_BN;
  const int kb = sh == SHAPE_FULL && !ep.logit_V ? KB_FULL : 128;
  CUtensorMap ta, tb, tc;
  if (!make_kmajor_map(&ta, A, K, M, lda, BM, kb) || !make_kmajor_map(&tb, B, K, N, ldb, b_box_rows(bn), kb) ||
      !make_map(&tc, ep.out, 2, ep.ldo, M, ep.ldo, 64, 32))
    return cudaErrorInvalidValue;
  if (ep.logit_V) {
    // the Performance-Optimized step's forward (never narrowed)
    if (!ep.zpart || ep.logit_ldV < N || ep.narrow) return cudaErrorInvalidValue;
    if (sh == SHAPE_FULL)
      return launch_tc<FWD_BN, false, false, MODE_FWD_LOGITS, USE_PAIR, NSTAGES, ROW_SUBTILES>(ta, tb, tc, 1, M, N, K,
                                                                                               ep, err, st);
    return launch_tc<FWD_BN, false, false, MODE_FWD_LOGITS, USE_PAIR, NSTAGES_SMALL, 1>(ta, tb, tc, 1, M, N, K, ep, err,
                                                                                        st);
  }
  if (sh == SHAPE_TINY)
    return launch_tc<TINY_BN, false, false, MODE_FWD, USE_PAIR, NSTAGES_TINY, 1>(ta, tb, tc, 1, M, N, K, ep, err, st);
  if (sh == SHAPE_SMALL)
    return launch_tc<FWD_BN, false, false, MODE_FWD, USE_PAIR, NSTAGES_SMALL, 1>(ta, tb, tc, 1, M, N, K, ep, err, st);
  return launch_tc<FWD_BN, false, false, MODE_FWD, USE_PAIR, NSTAGES_FULL, ROW_SUBTILES, 1, 2, KB_FULL>(ta, tb, tc, 1, M,
                                                                                                     N, K, ep, err, st);
}

// fp32 C written through shared memory and TMA when its rows are 16-byte
// aligned, directly otherwise.
static bool store_map(CUtensorMap* tc, float* C, int ldc, int rows, int cols) {
  return make_map(tc, C, 4, ldc, rows, ldc, 32, 32) && cols <= ldc;
}

cudaError_t tc_gemm_store(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K, float* Cm,
                          int ldc, int* err, cudaStream_t st) {
  const bool full = shape_of(M, N, FWD_BN) == SHAPE_FULL;
  const int kb = full ? KB_FULL : 128;
  CUtensorMap ta, tb, tc;
  if (!make_kmajor_map(&ta, A, K, M, lda, BM, kb) || !make_kmajor_map(&tb, B, K, N, ldb, b_box_rows(FWD_BN), kb))
    return cudaErrorInvalidValue;
  const int tma = store_map(&tc, Cm, ldc, M, N) ? 1 : 0;
  if (!tma) tc = ta;  // unused
  EpiArgs ep{nullptr, nullptr, Cm, ldc, nullptr};
  if (!full)
    return launch_tc<FWD_BN, false, false, MODE_STORE, USE_PAIR, NSTAGES_SMALL, 1>(ta, tb, tc, tma, M, N, K, ep, err,
                                                                                   st);
  return launch_tc<FWD_BN, false, false, MODE_STORE, USE_PAIR, NSTAGES_FULL, ROW_SUBTILES, 1, 2, KB_FULL>(
      ta, tb, tc, tma, M, N, K, ep, err, st);
}

cudaError_t tc_gemm_wgrad(const bf16* G, int ldg, const bf16* X, int ldx, int R, int N, int K, float* Cm, int ldc,
                          int* err, cudaStream_t st) {
  // C[N, K] = sum_r G[r, n] X[r, k]: the GEMM's M is N (rows of dW), its N is
  // K (columns of dW), its contraction is R; both operands MN-major.
  // MN-major boxes: 64 elements (128 bytes, 128-byte swizzle) of M or N by
  // one stage's K rows
  const bool full = shape_of(N, K, WGRAD_BN) == SHAPE_FULL;
  const int bke = (full ? KB_FULL : 128) / 2;
  CUtensorMap ta, tb, tc;
  if (!make_map(&ta, G, 2, N, R, ldg, 64, bke) || !make_map(&tb, X, 2, K, R, ldx, 64, bke))
    return cudaErrorInvalidValue;
  const int tma = store_map(&tc, Cm, ldc, N, K) ? 1 : 0;
  if (!tma) tc = ta;
  EpiArgs ep{nullptr, nullptr, Cm, ldc, nullptr};
  if (!full)
    return launch_tc<WGRAD_BN, true, true, MODE_STORE, USE_PAIR, NSTAGES_SMALL, 1>(ta, tb, tc, tma, N, K, R, ep, err,
                                                                                   st);
  return launch_tc<WGRAD_BN, true, true, MODE_STORE, USE_PAIR, NSTAGES_FULL, ROW_SUBTILES, 1, 2, KB_FULL>(
      ta, tb, tc, tma, N, K, R, ep, err, st);
}

// ------------------------------------------------ fp32 operands (3 x TF32)
// Stages of fp32 tiles with their lo parts: 96 KB with two 128-row subtiles
// per CTA (2 fit), 64 KB with one (3 fit).
constexpr int NSTAGES_F32 = 2;
constexpr int NSTAGES_F32_SMALL = 3;

bool tc_f32_supported(int K, int lda, int ldb) {
  // TMA rows of 16-byte multiples: fp32 row strides and K in multiples of 4
  return tc_supported() && (K & 3) == 0 && (lda & 3) == 0 && (ldb & 3) == 0;
}

cudaError_t tc_gemm_fwd_f32(const float* A, int lda, const float* B, int ldb, int M, int N, int K, const EpiArgs& ep,
                            int* err, cudaStream_t st) {
  if (!tc_f32_supported(K, lda, ldb) || ep.logit_V || ep.gpart_in || (ep.ldo & 3)) return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tc;
  if (!make_map(&ta, A, 4, K, M, lda, 32, BM) || !make_map(&tb, B, 4, K, N, ldb, 32, b_box_rows(FWD_BN)) ||
      !make_map(&tc, ep.out, 4, ep.ldo, M, ep.ldo, 32, 32))
    return cudaErrorInvalidValue;
  if (shape_of(M, N, FWD_BN) != SHAPE_FULL)
    return launch_tc<FWD_BN, false, false, MODE_FWD, USE_PAIR, NSTAGES_F32_SMALL, 1, 1, 4>(ta, tb, tc, 1, M, N, K, ep,
                                                                                          err, st);
  return launch_tc<FWD_BN, false, false, MODE_FWD, USE_PAIR, NSTAGES_F32, ROW_SUBTILES, 1, 4>(ta, tb, tc, 1, M, N, K,
                                                                                              ep, err, st);
}

cudaError_t tc_gemm_store_f32(const float* A, int lda, const float* B, int ldb, int M, int N, int K, float* Cm,
                              int ldc, int* err, cudaStream_t st) {
  if (!tc_f32_supported(K, lda, ldb)) return cudaErrorInvalidValue;
  CUtensorMap ta, tb, tc;
  if (!make_map(&ta, A, 4, K, M, lda, 32, BM) || !make_map(&tb, B, 4, K, N, ldb, 32, b_box_rows(FWD_BN)))
    return cudaErrorInvalidValue;
  const int tma = store_map(&tc, Cm, ldc, M, N) ? 1 : 0;
  if (!tma) tc = ta;  // unused
  EpiArgs ep{nullptr, nullptr, Cm, ldc, nullptr};
  if (shape_of(M, N, FWD_BN) != SHAPE_FULL)
    return launch_tc<FWD_BN, false, false, MODE_STORE, USE_PAIR, NSTAGES_F32_SMALL, 1, 1, 4>(ta, tb, tc, tma, M, N, K,
                                                                                            ep, err, st);
  return launch_tc<FWD_BN, false, false, MODE_STORE, USE_PAIR, NSTAGES_F32, ROW_SUBTILES, 1, 4>(ta, tb, tc, tma, M, N,
                                                                                                K, ep, err, st);
}

}  // namespace ff
