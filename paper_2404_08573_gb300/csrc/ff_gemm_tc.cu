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

// At most 96 registers a thread (the bound for two CTAs of 320 threads per
// SM; no spills): a CTA then leaves room on its SM for the Adam and local-
// gradient blocks of the other layers' streams (784-2000x4 epoch -1 %).
// MODE_FWD_LG: tmD maps dZ' (as tmC maps H) and lg holds the local step's
// arguments; the grid's column tiles all lie in one cluster (2 x gridDim.y).
template <int BN, bool A_MN, bool B_MN, int MODE, bool PAIR, int NSTAGE, int MT, int NT, int OPB, int KB>
__global__ void __launch_bounds__(NTHREADS, 2)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmD, int tma_store, int M,
              int N, int K, EpiArgs ep, GradPrepArgs lg, int* err) {
  using C = TcCfg<BN, NSTAGE, MT, PAIR, NT, OPB, KB>;
  constexpr bool FWD = MODE != MODE_STORE;
  constexpr bool LOGITS = MODE == MODE_FWD_LOGITS;
  constexpr bool LG = MODE == MODE_FWD_LG;
  constexpr bool TF32 = OPB == 4;
  static_assert(!TF32 || (!A_MN && !B_MN && (MODE == MODE_FWD || MODE == MODE_STORE)),
                "fp32 operands: K-major forward and store GEMMs");
  static_assert(KB == 128 || (MODE == MODE_FWD || MODE == MODE_STORE), "64-byte K rows: plain forward and store");
  static_assert(!LG || (PAIR && MT == 1 && NT == 2 && BN == 256 && EPI_WARPS == 8),
                "the local-gradient epilogue: 128 rows x 512 columns per CTA, a warp per 32 rows x 256 columns");
  // Block logits on the tensor cores (one 128-row subtile per CTA leaves TMEM
  // room for them): per column half, a pair MMA of the staged bf16 activity
  // (M = 256 across the pair, K = 128) with the block's weights (N = 16
  // classes, 8 per CTA, as a hi and a lo bf16 part) into 16 spare TMEM
  // columns.  With two subtiles the CUDA cores form them (10 fmas an element).
  constexpr bool LMMA = LOGITS && PAIR && MT == 1 && NT == 1 && BN == 256 && EPI_WARPS == 8;
  constexpr uint32_t TCOLS = LMMA ? 512 : C::TMEM_COLS;  // + the logits' 2 x 16 columns (a power of 2)
  constexpr uint32_t LCOL = MT * NT * C::ACC_COLS;       // first logits column
  extern __shared__ uint8_t smem_raw[];
  // 128-byte swizzled tiles need 1024-byte aligned shared addresses.
  const uint32_t raw_s = ptx::smem_u32(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_s & 1023u)) & 1023u);
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  // fp32: the lo parts of A and B, at the same offsets one ring further on
  constexpr int LO = C::STAGES * C::IN_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(tfull + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tslot + 1);
  volatile int* never_set = reinterpret_cast<volatile int*>(tslot + 2);  // drain waits ignore the abort
  volatile int* lgiss = reinterpret_cast<volatile int*>(tslot + 3);     // LMMA: bit h, half h's MMAs issued
  uint64_t* lgbar = reinterpret_cast<uint64_t*>(tslot + 4);  // LG: every partial of the row block has arrived
  uint64_t* conv = lgbar + 1;  // fp32: [STAGES] both CTAs' splits of a stage are done
  uint64_t* hst = conv + C::STAGES;  // LMMA: [2] both CTAs' activity of a column half is staged
  uint64_t* lgd = hst + 2;           // LMMA: [2] that half's logits MMAs are done
  float* sbias = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(full) + 256);  // [TN] bias of this tile
  float* sVt = sbias + C::TN;  // LOGITS: [BN][kLogitStride] block weights of this tile's columns
  // LMMA: the weights as MMA operands, 1024-byte aligned after the bias:
  // [half][hi, lo][64-column atom] tiles of 8 classes x 128 bytes
  uint8_t* sVb = reinterpret_cast<uint8_t*>(full) + 2048;
  // LG: [kLgParts][MT * BM] goodness partials of this CTA's rows (partial t
  // covers columns 128t ..), then per epilogue warp [2][32] row terms
  float* sgp = sbias + C::TN;
  float* scc = sgp + kLgParts * MT * BM;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // blockIdx.x: row tile (the two CTAs of a pair are consecutive in x, as
  // cta_group::2 requires); blockIdx.y: column tile
  const int m0 = blockIdx.x * (BM * MT);
  const int n0 = blockIdx.y * C::TN;
  const int num_kb = (K + C::BKE - 1) / C::BKE;

  // PAIR: the two CTAs of a cluster (consecutive tile rows, same columns)
  // compute their 2 x MT x BM rows with cta_group::2 MMAs (M = 256).  Each
  // CTA loads its own A rows and half of the B tile (columns crank*BN/2 ..);
  // with one 128-row subtile a CTA moves 32 KB per 64-deep K step for
  // 4.2 MFLOP instead of 48 KB for the same tile alone.  The
  // even CTA issues the MMAs once both halves of a stage have landed (the odd
  // CTA's copies complete on the even CTA's `full` barrier) and its commits
  // arrive on both CTAs' `empty` and `tfull` barriers.
  // A cluster may hold several pairs (LG: a pair per column tile); the pair
  // is the two CTAs whose cluster ranks differ in bit 0.
  uint32_t crank = 0;
  if constexpr (PAIR) crank = ptx::cluster_ctarank();
  const uint32_t pair_lead = crank & ~1u;
  const bool issuer = !PAIR || (crank & 1u) == 0;
  const uint16_t pmask = (uint16_t)(3u << pair_lead);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    ptx::mbar_init(tfull, 1);
    if constexpr (LG) ptx::mbar_init(lgbar, 32 * EPI_WARPS * gridDim.y);  // every epilogue lane of the row block
    if constexpr (TF32)
      for (int s = 0; s < C::STAGES; ++s) ptx::mbar_init(&conv[s], (PAIR ? 2 : 1) * EPI_WARPS);
    if constexpr (LMMA)
      for (int h = 0; h < 2; ++h) {
        ptx::mbar_init(&hst[h], 2 * (EPI_WARPS / 2));  // the 4 warps of the half in each CTA
        ptx::mbar_init(&lgd[h], 1);
      }
    *abort_flag = 0;
    *never_set = 0;
    *lgiss = 0;
    ptx::fence_mbar_init();
    ptx::prefetch_tmap(&tmA);
    ptx::prefetch_tmap(&tmB);
    if (FWD || tma_store) ptx::prefetch_tmap(&tmC);
    if constexpr (LG) ptx::prefetch_tmap(&tmD);
  }
  if (warp == 1) {
    if constexpr (PAIR) {
      ptx::tmem_alloc_pair(tslot, TCOLS);
      ptx::tmem_relinquish_pair();
    } else {
      ptx::tmem_alloc(tslot, TCOLS);
      ptx::tmem_relinquish();
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) ptx::cluster_sync();  // both CTAs' barriers and TMEM exist before any cross-CTA use
  ptx::tc_fence_after();
  const uint32_t tmem = *tslot;
  // everything above touched only this CTA's own resources: the inputs are
  // read, and the outputs written, only after the previous kernel is done
  ptx::griddep_wait();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      // the stage barriers the copies complete on: the issuing CTA's
      uint32_t full0 = ptx::smem_u32(&full[0]);
      if constexpr (PAIR) full0 = ptx::mapa_shared(full0, pair_lead);
      auto load = [&](void* dst, const CUtensorMap* map, int s, int c0, int c1) {
        if (!ff_dcheck(tma_x_aligned(c0, OPB), err)) {
          *abort_flag = 1;
          return;
        }
        // fp32: each CTA's copies complete on its own barrier (its epilogue
        // warps split them before the pair's MMAs read them)
        if constexpr (PAIR && !TF32)
          ptx::tma_load_2d_pair(dst, map, full0 + 8u * (uint32_t)s, c0, c1);
        else
          ptx::tma_load_2d(dst, map, &full[s], c0, c1);
      };
      const int nb = n0 + (int)(crank & 1u) * C::BH;  // first B column this CTA loads (of column subtile 0)
      int issued = 0;
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % C::STAGES;
        const uint32_t ph = (uint32_t)(kb / C::STAGES) & 1u;
        if (!ptx::mbar_wait(&empty[s], ph ^ 1u, kWaitTimeoutNs, abort_flag)) {
          latch(err, abort_flag);
          break;
        }
        if constexpr (TF32)
          ptx::mbar_arrive_expect_tx(&full[s], C::IN_BYTES);
        else if (issuer)
          ptx::mbar_arrive_expect_tx(&full[s], PAIR ? 2 * C::STAGE : C::STAGE);
        uint8_t* a = sA + s * C::A_BYTES;
        uint8_t* b = sB + s * C::B_BYTES;
        const int k0 = kb * C::BKE;
        if (!A_MN) {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) load(a + mt * BM * C::KBYTES, &tmA, s, k0, m0 + BM * mt);
        } else {
#pragma unroll
          for (int j = 0; j < MT * BM / 64; ++j) load(a + j * 64 * C::BKE * 2, &tmA, s, m0 + 64 * j, k0);
        }
        if (!B_MN) {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) load(b + nt * C::BH * C::KBYTES, &tmB, s, k0, nb + nt * BN);
        } else {
#pragma unroll
          for (int j = 0; j < C::BH / 64; ++j) load(b + j * 64 * C::BKE * 2, &tmB, s, nb + 64 * j, k0);
        }
        issued = kb + 1;
      }
      if (PAIR && !*abort_flag) {
        // Producer tail: wait for the commits of the last stages, so that no
        // arrival from the other CTA targets this one after it exits.
        for (int kb = num_kb; kb < num_kb + C::STAGES; ++kb) {
          if (!ptx::mbar_wait(&empty[kb % C::STAGES], ((uint32_t)(kb / C::STAGES) & 1u) ^ 1u, kWaitTimeoutNs,
                              abort_flag)) {
            latch(err, abort_flag);
            break;
          }
        }
      }
      if (*abort_flag) {
        if (issuer || TF32) {
          // let copies already issued land before the CTA's shared memory goes away
          int lo = issued - C::STAGES;
          if (lo < 0) lo = 0;
          for (int kb = lo; kb < issued; ++kb)
            ptx::mbar_wait(&full[kb % C::STAGES], (uint32_t)(kb / C::STAGES) & 1u, 10000000ull, never_set);
        } else {
          // this CTA's copies complete on the other CTA's barrier: give them
          // time to land
          const uint64_t t0 = ptx::globaltimer();
          while (ptx::globaltimer() - t0 < 1000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0 && issuer) {
      constexpr uint32_t idesc = TF32 ? ptx::idesc_tf32_f32(PAIR ? 2 * BM : BM, BN)
                                      : ptx::idesc_bf16_f32(PAIR ? 2 * BM : BM, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % C::STAGES;
        const uint32_t ph = (uint32_t)(kb / C::STAGES) & 1u;
        // fp32: the stage is split in both CTAs (remote arrivals: cluster-scope acquire)
        const bool ready = TF32 ? ptx::mbar_wait_cluster(&conv[s], ph, kWaitTimeoutNs, abort_flag)
                                : ptx::mbar_wait(&full[s], ph, kWaitTimeoutNs, abort_flag);
        if (!ready) {
          latch(err, abort_flag);
          break;
        }
        ptx::tc_fence_after();
        const uint32_t a_base = ptx::smem_u32(sA + s * C::A_BYTES);
        const uint32_t b_base = ptx::smem_u32(sB + s * C::B_BYTES);
#pragma unroll
        for (int k = 0; k < C::KBYTES / 32; ++k) {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            // K-major: the 32-byte K slice of one MMA sits 32 bytes further
            // along each swizzled row (SBO = 8 rows: 1024 bytes with 128-byte
            // rows, 512 with 64-byte ones).  MN-major: 16 K rows further = 2 x
            // 1024 bytes; LBO = 128 x BKE between the 64-element MN chunks,
            // SBO = 1024 between 8-row K groups.  Column subtile nt: its own B
            // box, BH rows further.
            const uint32_t bs = b_base + nt * C::BH * C::KBYTES;
            const uint64_t bd = B_MN            ? ptx::sdesc_sw128(bs + k * 2048, 64 * C::BKE * 2, 1024)
                                : KB == 128     ? ptx::sdesc_sw128(bs + k * 32, 16, 1024)
                                                : ptx::sdesc_sw64(bs + k * 32, 16, 512);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              // row subtile mt: BM rows further in the A stage, its own accumulator
              const uint32_t as = a_base + mt * BM * C::KBYTES;
              const uint64_t ad = A_MN        ? ptx::sdesc_sw128(as + k * 2048, 64 * C::BKE * 2, 1024)
                                  : KB == 128 ? ptx::sdesc_sw128(as + k * 32, 16, 1024)
                                              : ptx::sdesc_sw64(as + k * 32, 16, 512);
              const uint32_t acc = tmem + (uint32_t)((mt * NT + nt) * C::ACC_COLS);
              if constexpr (TF32) {
                // Ah Bh + Ah Bl + Al Bh (the lo parts LO bytes further on)
                const uint64_t adl = ptx::sdesc_sw128(as + LO + k * 32, 16, 1024);
                const uint64_t bdl = ptx::sdesc_sw128(bs + LO + k * 32, 16, 1024);
                if constexpr (PAIR) {
                  ptx::umma_tf32_pair(acc, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
                  ptx::umma_tf32_pair(acc, ad, bdl, idesc, 1u);
                  ptx::umma_tf32_pair(acc, adl, bd, idesc, 1u);
                } else {
                  ptx::umma_tf32(acc, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
                  ptx::umma_tf32(acc, ad, bdl, idesc, 1u);
                  ptx::umma_tf32(acc, adl, bd, idesc, 1u);
                }
              } else if constexpr (PAIR) {
                ptx::umma_f16_pair(acc, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
              } else {
                ptx::umma_f16(acc, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
              }
            }
          }
        }
        if constexpr (PAIR)
          ptx::umma_commit_pair(&empty[s], pmask);
        else
          ptx::umma_commit(&empty[s]);
      }
      // always: the epilogues and the teardown wait on it
      if constexpr (PAIR)
        ptx::umma_commit_pair(tfull, pmask);
      else
        ptx::umma_commit(tfull);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // Warp w (2..9) reads TMEM lane quarter q = w % 4 -- row 32q + t of each
    // of the MT row subtiles for its thread t -- and the columns of half
    // (w - 2) / 4 of the tile.  The operand ring is idle once the
    // accumulators are complete, so each warp stages its block there in the
    // 128-byte-swizzled layout (conflict-free for row-per-thread 16-byte
    // writes) and one lane writes it out with TMA.
    constexpr int HALVES = EPI_WARPS / 4;
    constexpr int CPW = C::TN / HALVES;  // columns per epilogue warp (within one accumulator)
    const int q = warp & 3;
    const int ew = warp - 2;          // 0 .. EPI_WARPS-1
    const int half = ew / 4;
    const int cbase = half * CPW;     // this warp's first column within the tile
    float srow[MT];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) srow[mt] = 0.f;
    if (FWD) {
      // While the mainloop runs: the tile's bias (zero past N or without bias)
      // into shared memory and this thread's row scales into registers.
      for (int c = (int)threadIdx.x - 64; c < C::TN; c += 32 * EPI_WARPS)
        sbias[c] = (ep.bias != nullptr && n0 + c < N) ? __ldg(ep.bias + n0 + c) : 0.f;
      if constexpr (LMMA) {
        // this CTA's 8 classes (the pair splits the 16 padded classes of the
        // MMA's N) of the tile's 256 columns, as bf16 hi = rn(v) and
        // lo = rn(v - hi), in 128-byte-swizzled K-major tiles
        const int cl0 = 8 * (int)(crank & 1u);
        for (int idx = (int)threadIdx.x - 64; idx < 2 * 2 * 8 * 64; idx += 32 * EPI_WARPS) {
          const int j = idx & 63, i = (idx >> 6) & 7, a = (idx >> 9) & 1, h = idx >> 10;
          const int cl = cl0 + i, col = n0 + h * 128 + a * 64 + j;
          const float v = cl < kLogitClasses && col < N ? __ldg(ep.logit_V + (size_t)cl * ep.logit_ldV + col) : 0.f;
          const bf16 hi = __float2bfloat16_rn(v);
          const bf16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
          const int off = i * 128 + (((j >> 3) ^ (i & 7)) << 4) + (j & 7) * 2;
          *reinterpret_cast<bf16*>(sVb + ((h * 2 + 0) * 2 + a) * 1024 + off) = hi;
          *reinterpret_cast<bf16*>(sVb + ((h * 2 + 1) * 2 + a) * 1024 + off) = lo;
        }
        ptx::fence_async_smem();  // read by the logits MMAs (async proxy)
      } else if constexpr (LOGITS) {
        for (int idx = (int)threadIdx.x - 64; idx < kLogitClasses * BN; idx += 32 * EPI_WARPS) {
          const int c = idx / BN, j = idx % BN;
          sVt[j * kLogitStride + c] = n0 + j < N ? __ldg(ep.logit_V + (size_t)c * ep.logit_ldV + n0 + j) : 0.f;
        }
      }
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        const int gi = m0 + mt * BM + q * 32 + lane;
        if (gi >= M) continue;
        if (ep.gpart_in) {
          const float gprev = sum_partials(ep.gpart_in, ep.ntiles_in, M, gi);
          srow[mt] = inv_norm(gprev);
          if (blockIdx.y == 0 && half == 0) {  // one thread per row
            if (!isfinite(gprev)) atomicOr(err, DEVERR_NONFINITE);
            if (ep.G_acc) ep.G_acc[gi] += gprev;
            if (ep.s_out) ep.s_out[gi] = srow[mt];
          }
        } else {
          srow[mt] = __ldg(ep.row_scale + gi);
        }
      }
      ptx::named_bar(1, 32 * EPI_WARPS);
    }
    if constexpr (TF32) {
      // Split every stage this CTA receives: x -> xh = x with the 13 low
      // mantissa bits cleared (in place), xl = x - xh (LO bytes further on);
      // then one arrival per warp on the pair's (even CTA's) barrier.
      constexpr int V4 = C::IN_BYTES / 16;  // 16-byte words per stage
      const int t = (int)threadIdx.x - 64;
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % C::STAGES;
        const uint32_t ph = (uint32_t)(kb / C::STAGES) & 1u;
        const bool got = ptx::mbar_wait(&full[s], ph, kWaitTimeoutNs, abort_flag);
        if (!got) latch(err, abort_flag);
        if (!__all_sync(0xffffffffu, got && !*abort_flag)) break;
        // the stage's A and B boxes: A_BYTES at sA + s A_BYTES, B_BYTES at sB + s B_BYTES
        for (int i = t; i < V4; i += 32 * EPI_WARPS) {
          const int byte = i * 16;
          uint8_t* p = byte < C::A_BYTES ? sA + s * C::A_BYTES + byte : sB + s * C::B_BYTES + (byte - C::A_BYTES);
          uint4 x = *reinterpret_cast<uint4*>(p);
          uint4 h, l;
          h.x = x.x & 0xFFFFE000u; h.y = x.y & 0xFFFFE000u; h.z = x.z & 0xFFFFE000u; h.w = x.w & 0xFFFFE000u;
          l.x = __float_as_uint(__fsub_rn(__uint_as_float(x.x), __uint_as_float(h.x)));
          l.y = __float_as_uint(__fsub_rn(__uint_as_float(x.y), __uint_as_float(h.y)));
          l.z = __float_as_uint(__fsub_rn(__uint_as_float(x.z), __uint_as_float(h.z)));
          l.w = __float_as_uint(__fsub_rn(__uint_as_float(x.w), __uint_as_float(h.w)));
          *reinterpret_cast<uint4*>(p) = h;
          *reinterpret_cast<uint4*>(p + LO) = l;
        }
        ptx::fence_async_smem();  // the MMAs (async proxy) read what these generic writes left
        __syncwarp();
        if (lane == 0) {
          if (issuer)
            ptx::mbar_arrive(&conv[s]);
          else
            ptx::mbar_arrive_remote(&conv[s], pair_lead);
        }
      }
    }
    const bool ok = ptx::mbar_wait(tfull, 0, kWaitTimeoutNs, abort_flag);
    if (threadIdx.x == 64) ptx::griddep_launch_dependents();  // the mainloop is done
    if (!ok) latch(err, abort_flag);
    ptx::tc_fence_after();
    // tcgen05.ld is warp-collective: decide for the whole warp at once
    if (__all_sync(0xffffffffu, ok && !*abort_flag)) {
      constexpr int ES = FWD && !TF32 ? 2 : 4;  // staged element size (the output's)
      constexpr int CW = 128 / ES;                       // columns per 128-byte swizzle row
      const uint32_t sw = (uint32_t)(lane & 7);
      const bool staged = FWD || tma_store;
      int fchunk = 0;  // fp32 chunks streamed so far (slot parity)
#pragma unroll 1
      for (int mt = 0; mt < MT; ++mt) {
        const int rbase = m0 + mt * BM + q * 32;  // this warp's first row in subtile mt
        const int gi = rbase + lane;
        // bf16: the warp's 32 x CPW block per subtile; fp32: two 32 x 32 slots, streamed
        uint8_t* stage = smem + (FWD && !TF32 ? (ew * MT + mt) * (32 * CPW * 2) : ew * 8192);
        // the warp's 32 rows of its 64-column chunk ch of the activity; LMMA:
        // inside the half's 128-row swizzle atoms (the logits MMA's A operand)
        auto chunk = [&](int ch) -> uint8_t* {
          if constexpr (LMMA) return smem + (half * 2 + ch) * 16384 + q * 32 * 128;
          return stage + ch * (32 * 128);
        };
        const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) +
                              (uint32_t)((mt * NT + cbase / BN) * C::ACC_COLS + cbase % BN);
        const float s = srow[mt];
        float g = 0.f;
        float g_lo = 0.f;  // LG: the goodness partial of the warp's first 128 columns
        float zl[kLogitClasses];  // LOGITS: this row's partial logits over the warp's columns
#pragma unroll
        for (int c = 0; c < kLogitClasses; ++c) zl[c] = 0.f;
        // Columns past N and rows past M hold zero products (their operand rows
        // were zero-filled); the TMA store clips them and gpart skips them.
        // c0 counts columns within this warp's half.
        auto process = [&](const uint32_t (&r)[32], int c0) {
          const int col0 = n0 + cbase + c0;
          if (FWD && !TF32) {
            uint32_t packed[16];
            const float4* b4 = reinterpret_cast<const float4*>(sbias + cbase + c0);
#pragma unroll
            for (int v = 0; v < 8; ++v) {
              const float4 bb = b4[v];
              const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
              float h[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float z = fmaf(s, __uint_as_float(r[4 * v + e]), bv[e]);
                h[e] = z != z ? z : fmaxf(z, 0.f);  // ReLU, NaN kept for the non-finite check
                g = fmaf(h[e], h[e], g);
              }
              __nv_bfloat162 p0 = __floats2bfloat162_rn(h[0], h[1]);
              __nv_bfloat162 p1 = __floats2bfloat162_rn(h[2], h[3]);
              packed[2 * v] = *reinterpret_cast<uint32_t*>(&p0);
              packed[2 * v + 1] = *reinterpret_cast<uint32_t*>(&p1);
              if constexpr (LOGITS && !LMMA) {
                // the block reads the stored (bf16-rounded) activity
                const float2 lo = __bfloat1622float2(p0), hi = __bfloat1622float2(p1);
                const float hr[4] = {lo.x, lo.y, hi.x, hi.y};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float4* vt = reinterpret_cast<const float4*>(sVt + (cbase + c0 + 4 * v + e) * kLogitStride);
                  const float4 v0 = vt[0], v1 = vt[1], v2 = vt[2];
                  const float vv[kLogitClasses] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w, v2.x, v2.y};
#pragma unroll
                  for (int c = 0; c < kLogitClasses; ++c) zl[c] = fmaf(hr[e], vv[c], zl[c]);
                }
              }
            }
            uint8_t* base = chunk(c0 / CW) + lane * 128;
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const uint32_t j = (uint32_t)((c0 % CW) / 8 + v);
              *reinterpret_cast<uint4*>(base + ((j ^ sw) << 4)) =
                  make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2], packed[4 * v + 3]);
            }
          } else if (staged) {
            // fp32: chunk n goes through slot n&1; before refilling a slot the
            // store issued from it two chunks ago must have read it
            uint8_t* sbuf = stage + (fchunk & 1) * 4096;
            if (lane == 0 && fchunk >= 2) ptx::bulk_wait_read1();
            __syncwarp();
            uint8_t* base = sbuf + lane * 128;
#pragma unroll
            for (int v = 0; v < 8; ++v) {
              uint32_t o[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                if constexpr (FWD) {
                  // fp32 forward: the activity itself, and its goodness
                  const float z = fmaf(s, __uint_as_float(r[4 * v + e]), sbias[cbase + c0 + 4 * v + e]);
                  const float h = z != z ? z : fmaxf(z, 0.f);
                  g = fmaf(h, h, g);
                  o[e] = __float_as_uint(h);
                } else {
                  o[e] = r[4 * v + e];
                }
              }
              *reinterpret_cast<uint4*>(base + (((uint32_t)v ^ sw) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
            }
            ptx::fence_async_smem();
            __syncwarp();
            if (lane == 0 && rbase < M && col0 < ep.ldo &&
                ff_dcheck(col0 >= 0 && rbase >= 0 && tma_x_aligned(col0, 4), err))
              ptx::tma_store_2d(&tmC, sbuf, col0, rbase);
            if (lane == 0) ptx::bulk_commit();
            ++fchunk;
          } else if (gi < M) {
            float* out = reinterpret_cast<float*>(ep.out) + (size_t)gi * ep.ldo;
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (col0 + j < N) out[col0 + j] = __uint_as_float(r[j]);
          }
        };
        // TMEM loads double-buffered: the next 32 columns load while these are processed.
        uint32_t ra[32], rb[32];
        ptx::tmem_ld32(trow, ra);
        ptx::tmem_ld_wait();
#pragma unroll 1
        for (int c0 = 0; c0 < CPW; c0 += 64) {
          ptx::tmem_ld32(trow + (uint32_t)(c0 + 32), rb);
          process(ra, c0);
          ptx::tmem_ld_wait();
          if (c0 + 64 < CPW) ptx::tmem_ld32(trow + (uint32_t)(c0 + 64), ra);
          process(rb, c0 + 32);
          ptx::tmem_ld_wait();
          if constexpr (LG) {
            // partials per 128 columns, as the tile shapes of the other forms give
            if (c0 + 64 == 128) {
              g_lo = g;
              g = 0.f;
            }
          }
        }
        if (FWD && !LG && gi < M) ep.gpart[(size_t)(blockIdx.y * HALVES + half) * M + gi] = g;
        if (LOGITS && !LMMA && gi < M) {
          float2* zp = reinterpret_cast<float2*>(ep.zpart + ((size_t)(blockIdx.y * HALVES + half) * M + gi) * kLogitClasses);
#pragma unroll
          for (int c = 0; c < kLogitClasses; c += 2) zp[c / 2] = make_float2(zl[c], zl[c + 1]);
        }
        if (FWD && !TF32) {
          ptx::fence_async_smem();
          __syncwarp();
          if (lane == 0 && rbase < M) {
#pragma unroll 1
            for (int ch = 0; ch < CPW / CW; ++ch) {
              const int col = n0 + cbase + ch * CW;
              if (col < ep.ldo && ff_dcheck(col >= 0 && rbase >= 0 && tma_x_aligned(col, 2), err))
                ptx::tma_store_2d(&tmC, chunk(ch), col, rbase);
            }
            ptx::bulk_commit();
          }
        }
        if constexpr (LMMA) {
          // The block's partial logits of this half: once the 4 warps of the
          // half have staged their rows in both CTAs, one thread of the even
          // CTA issues the pair MMAs (K = 128 as 8 steps of 16, the weights'
          // hi and lo parts), committed to both CTAs' barrier.
          if (lane == 0) {
            if (issuer)
              ptx::mbar_arrive(&hst[half]);
            else
              ptx::mbar_arrive_remote(&hst[half], pair_lead);
          }
          if (issuer && q == 0 && lane == 0) {
            if (ptx::mbar_wait_cluster(&hst[half], 0, kWaitTimeoutNs, abort_flag)) {
              ptx::tc_fence_after();
              constexpr uint32_t idesc_l = ptx::idesc_bf16_f32(2 * BM, 16, 0, 0);
#pragma unroll
              for (int sp = 0; sp < 2; ++sp)
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                  const uint32_t a_addr = ptx::smem_u32(smem + (half * 2 + (kk >> 2)) * 16384) + (kk & 3) * 32;
                  const uint32_t b_addr = ptx::smem_u32(sVb + ((half * 2 + sp) * 2 + (kk >> 2)) * 1024) + (kk & 3) * 32;
                  ptx::umma_f16_pair(tmem + LCOL + 16 * half, ptx::sdesc_sw128(a_addr, 16, 1024),
                                     ptx::sdesc_sw128(b_addr, 16, 1024), idesc_l, (sp | kk) != 0 ? 1u : 0u);
                }
              ptx::umma_commit_pair(&lgd[half], pmask);
              atomicOr(const_cast<int*>(lgiss), 1 << half);
            } else {
              latch(err, abort_flag);
            }
          }
          const bool done = ptx::mbar_wait(&lgd[half], 0, kWaitTimeoutNs, abort_flag);
          if (!done) latch(err, abort_flag);
          if (__all_sync(0xffffffffu, done && !*abort_flag)) {
            ptx::tc_fence_after();
            uint32_t rz[16];
            ptx::tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + LCOL + 16 * half, rz);
            ptx::tmem_ld_wait();
            if (gi < M) {
              float2* zp = reinterpret_cast<float2*>(ep.zpart +
                                                     ((size_t)(blockIdx.y * HALVES + half) * M + gi) * kLogitClasses);
#pragma unroll
              for (int c = 0; c < kLogitClasses; c += 2)
                zp[c / 2] = make_float2(__uint_as_float(rz[c]), __uint_as_float(rz[c + 1]));
            }
          }
        }
        if constexpr (LG) {
          // ---- the rest of the layer's local step (§3, Eq. 1) for the warp's
          // 32 rows x 256 columns, with every sum in the order of the separate
          // local-gradient kernel (k_grad_prep), so both give the same bits.
          const int r = q * 32 + lane;  // row within the CTA
          // (1) this warp's two partials into every CTA of the row block (this
          //     one included), then one arrival on each CTA's barrier
          {
            const int t0 = (n0 + cbase) / 128;
            const uint32_t xr = crank & 1u;
            for (uint32_t y = 0; y < gridDim.y; ++y) {
              const uint32_t rank = xr + 2u * y;
              ptx::st_remote_f32(&sgp[t0 * BM + r], rank, g_lo);
              ptx::st_remote_f32(&sgp[(t0 + 1) * BM + r], rank, g);
              ptx::mbar_arrive_remote(lgbar, rank);
            }
          }
          // (2) every partial of these rows has arrived (bounded)
          const bool have = ptx::mbar_wait_cluster(lgbar, 0, kWaitTimeoutNs, abort_flag);
          if (!have) latch(err, abort_flag);
          if (__all_sync(0xffffffffu, have && !*abort_flag)) {
            // (3) the row's goodness: 8 lane-strided sums over the partials
            //     (the ones past N are +0), then a fixed tree
            const int nparts = 4 * (int)gridDim.y;
            float gs[8];
#pragma unroll
            for (int p8 = 0; p8 < 8; ++p8) {
              float a = 0.f;
              for (int t = p8; t < nparts; t += 8) a += sgp[t * BM + r];
              gs[p8] = a;
            }
            const float gsum = ((gs[0] + gs[4]) + (gs[2] + gs[6])) + ((gs[1] + gs[5]) + (gs[3] + gs[7]));
            const bool row_ok = gi < M;
            const bool pos = gi < lg.B;
            const float tt = pos ? lg.theta - gsum : gsum - lg.theta;  // the pair member's margin error
            float cc = 0.f, sc = 0.f;  // 2 dL/dg, and times the row scale
            if (row_ok) {
              const float sg = sigmoid_f(tt);
              cc = 2.f * (pos ? -sg : sg) / (float)lg.B;
              sc = s * cc;
            }
            const bool lead = blockIdx.y == 0 && half == 0;  // one thread per row
            float lv = 0.f, gpv = 0.f, gnv = 0.f;
            if (lead && row_ok) {
              if (!isfinite(gsum)) atomicOr(err, DEVERR_NONFINITE);
              if (lg.g_out) lg.g_out[gi] = gsum;
              if (lg.s_next) lg.s_next[gi] = inv_norm(gsum);
              lv = softplus_f(tt);
              (pos ? gpv : gnv) = gsum;
            }
            float* ccw = scc + ew * 64;  // [32] 2 dL/dg, then [32] s 2 dL/dg of the warp's rows
            ccw[lane] = cc;
            ccw[32 + lane] = sc;
            const int rb = rbase / 32;  // the 32-row block
            const int nrb = (M + 31) / 32;
            if (lead) {
              // the block's loss and goodness sums: rows y, y+8, y+16, y+24 as
              // (y + (y+16)) + ((y+8) + (y+24)), then y = 0..7 in turn
              auto block_sum = [&](float v) {
                v += __shfl_down_sync(0xffffffffu, v, 16);
                v += __shfl_down_sync(0xffffffffu, v, 8);
                float t = 0.f;
#pragma unroll
                for (int y = 0; y < 8; ++y) t += __shfl_sync(0xffffffffu, v, y);
                return t;
              };
              const float tl = block_sum(lv), tp = block_sum(gpv), tn = block_sum(gnv);
              if (lane == 0 && rbase < M) {
                lg.loss_part[rb] = tl;
                if (lg.stat_part) {
                  lg.stat_part[rb] = tp;
                  lg.stat_part[nrb + rb] = tn;
                }
              }
              if (blockIdx.x == 0 && q == 0 && lane == 0 && lg.ds) {
                // the Adam update that follows is step t; beta^t as running products
                lg.ds->t += 1;
                lg.ds->pow1 *= lg.beta1;
                lg.ds->pow2 *= lg.beta2;
                lg.ds->bc1 = (float)(1.0 - lg.ds->pow1);
                lg.ds->bc2 = (float)(1.0 - lg.ds->pow2);
              }
            }
            // (4) once the activity's stores have read the staging, turn it in
            //     place into dZ' = bf16(s 2 dL/dg h) (h as stored; zero on rows
            //     past M), two columns per lane and pass: lane j takes columns
            //     64 p + 2j, +1, row by row -- conflict-free in the swizzled
            //     layout -- and forms their bias-gradient partials over the 32
            //     rows, db_y = chain of fmas over the rows y + 8k, then y = 0..7
            if (lane == 0) ptx::bulk_wait_read0();
            __syncwarp();
            float act = 0.f;
            const int nvalid = M - rbase;  // rows of the block below M
#pragma unroll 1
            for (int pass = 0; pass < CPW / 64; ++pass) {
              uint8_t* chunk = stage + pass * (32 * 128) + (lane & 3) * 4;
              float tA = 0.f, tB = 0.f;
#pragma unroll 2
              for (int y = 0; y < 8; ++y) {
                float dA = 0.f, dB = 0.f;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const int rr_ = y + 8 * k;
                  uint32_t* wp = reinterpret_cast<uint32_t*>(chunk + rr_ * 128 + ((((uint32_t)lane >> 2) ^ (uint32_t)(rr_ & 7)) << 4));
                  uint32_t w = *wp;
                  if (rr_ >= nvalid) w = 0u;
                  const float2 hf = __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&w));
                  const float cr = ccw[rr_], sr = ccw[32 + rr_];
                  dA = fmaf(cr, hf.x, dA);
                  dB = fmaf(cr, hf.y, dB);
                  act += (hf.x > 0.f ? 1.f : 0.f) + (hf.y > 0.f ? 1.f : 0.f);
                  __nv_bfloat162 zb = __floats2bfloat162_rn(sr * hf.x, sr * hf.y);
                  *wp = *reinterpret_cast<uint32_t*>(&zb);
                }
                tA += dA;
                tB += dB;
              }
              const int col = n0 + cbase + pass * 64 + 2 * lane;
              if (rbase < M) {
                if (col < N) lg.dbpart[(size_t)rb * N + col] = tA;
                if (col + 1 < N) lg.dbpart[(size_t)rb * N + col + 1] = tB;
              }
            }
            // (6) dZ' out with TMA, and the block's active-ReLU count
            ptx::fence_async_smem();
            __syncwarp();
            if (lane == 0 && rbase < M) {
#pragma unroll 1
              for (int ch = 0; ch < CPW / CW; ++ch) {
                const int col = n0 + cbase + ch * CW;
                if (col < ep.ldo && ff_dcheck(col >= 0 && rbase >= 0 && tma_x_aligned(col, 2), err))
                  ptx::tma_store_2d(&tmD, stage + ch * (32 * 128), col, rbase);
              }
              ptx::bulk_commit();
            }
            act = warp_sum(act);
            const int cb = (n0 + cbase) / 256;
            if (lane == 0 && lg.stat_part && cb < lg.ncb && rbase < M)
              lg.stat_part[2 * nrb + (size_t)rb * lg.ncb + cb] = act;
          }
        }
      }
      if (staged) {
        if (lane == 0) ptx::bulk_wait_read0();
        __syncwarp();
      }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) ptx::cluster_sync();  // both CTAs are done with the pair's TMEM and barriers
  ptx::tc_fence_after();
  if (warp == 1) {
    if (*abort_flag) {
      // MMAs issued before the abort must finish before TMEM is released
      ptx::mbar_wait(tfull, 0, 10000000ull, never_set);
      if constexpr (LMMA)
        for (int h = 0; h < 2; ++h) ptx::mbar_wait(&lgd[h], 0, 10000000ull, never_set);
    }
    if constexpr (PAIR)
      ptx::tmem_dealloc_pair(tmem, TCOLS);
    else
      ptx::tmem_dealloc(tmem, TCOLS);
  }
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
  static auto kernel() { return k_tc_gemm<BN, A_MN, B_MN, MODE, PAIR, NSTAGE, MT, NT, OPB, KB>; }
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
