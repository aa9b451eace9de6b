// Fused Z-panel contraction and dense loss pass on the tcgen05 tensor cores.
//
// For M-side rows m_i (a tile of 128) and Q-side rows q_k (streamed in
// chunks of BN), the panel kernel computes, without writing any tile of L or
// Z to global memory (the fused kernel of Sec. 4.2, eq. "kernel"):
//   L_ik = m_i . q_k                         MMA1: TMEM <- W tile x chunk^T
//   P_ik = min(0, L_ik)      (Z form, eq. updateZ)   -- epilogue in registers,
//        = -max(0, L_ik)     (Delta form, eq. updateD)  written back to TMEM
//   R_i  = sum_k P_ik q_k                    MMA2: TMEM R += P (TMEM) x chunk
// The same shared-memory copy of each chunk feeds both products: K-major for
// MMA1 and MN-major for MMA2.  The W tile is MMA1's A operand from shared
// memory (bf16 mode, TMA-loaded with the chunk's swizzle) or from TMEM
// (fp32-accurate mode, written by the epilogue warps).  Every factor has bf16 pieces hi = bf16(x),
// lo = bf16(x - hi), lo2 = bf16(x - hi - lo).  bf16 mode: MMA1 uses hi only,
// MMA2 uses q = hi + lo -- every row of R shares the same q_k, so a rounding
// of q would be a coherent error that the Gram solve amplifies by its
// condition number.  fp32-accurate mode (SPLIT): MMA1 = w_hi q_hi + w_hi q_lo
// + w_lo q_hi, P = P_hi + P_lo, MMA2 = P_hi (q_hi + q_lo + q_lo2) + P_lo q_hi.
//
// The loss kernel runs MMA1 only, over all of W against all of B, and sums
// max(0, L)^2 and max(0, L) over the entries outside the support of S (the
// dense parts of eq. SLloss / eq. RMSE / eq. WJD); the support entries are
// summed by a separate pass.
//
// Warp roles (352 threads, one CTA per SM, persistent over M tiles):
//   warps 0-7  epilogue, two warpgroups taking alternate chunks; in each,
//              thread t owns TMEM lane t = tile row t
//   warp 8     TMA producer of Q chunks and W tiles (+ TMEM allocation)
//   warp 9     issues MMA1 (L = W Q^T) for every chunk
//   warp 10    issues MMA2 (R += P Q) for every chunk
// The two MMA warps run converged and predicate each tcgen05 operation on an
// elected lane; with two issuers the bookkeeping of one (barrier polls,
// commits) overlaps the other's products on the tensor core.
// Every mbarrier wait is bounded (2 s): on expiry the kernel records
// NMD_ERR_TIMEOUT, the other roles stop at their next wait, in-flight MMAs
// and copies are drained and TMEM is freed before the kernel returns.
#include <cudaTypedefs.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <tuple>

#include "nmd_internal.cuh"
#include "tc_ptx.cuh"

namespace nmd {
namespace {

using namespace tc;

constexpr int kEpiThreads = 256;                 // two epilogue warpgroups
constexpr int kProducerWarp = 8, kMma1Warp = 9, kMma2Warp = 10;
constexpr int kThreads = 352;
constexpr int BM = 128;
constexpr uint64_t kTimeoutNs = 2000000000ull;

template <int RP, bool SPLIT, bool LOSS>
struct Cfg {
  // fp32-accurate mode at r_pad = 256: W hi + lo take 256 TMEM columns, so a
  // CTA accumulates one 128-column half of R (blockIdx.y selects it) and the
  // first product is formed once per half
  static constexpr bool RHALF = SPLIT && !LOSS && RP == 256;
  static constexpr int NR = RHALF ? RP / 2 : RP;        // R columns of one CTA
  // TMEM columns of the R accumulator; the loss pass has none.  In the bf16
  // mode the second product multiplies P by q_hi alone: the update pairs
  // this term with the Gram matrix of q_hi, so the rounding of q cancels
  // (see update_kernel), and R needs one accumulator of r_pad columns.
  static constexpr int RCOLS = LOSS ? 0 : NR;
  // bf16 mode, r_pad <= 128: the W tile is the first product's A operand
  // from shared memory (loaded by TMA) instead of TMEM, which leaves TMEM
  // to the L buffers.
  static constexpr bool WSMEM = !SPLIT && !LOSS && RP <= 128;
  // Q rows per chunk (the N of the first product and the K of the second):
  // 128 where three L buffers of 128 columns fit beside R (bf16 mode at
  // r_pad <= 64: 3 x 128 + r_pad <= 512); 64 where that would leave fewer
  // than three.  (Four buffers of 96 rows were slower at r_pad = 64.)
  static constexpr int BN = WSMEM ? (RP == 128 ? 64 : 128) : ((RP == 256 || (SPLIT && RP == 128)) ? 64 : 128);
  // TMEM columns of one W tile (hi [+ lo]); none when it sits in shared memory
  static constexpr int WCOLS = WSMEM ? 0 : (SPLIT ? RP : RP / 2);
  static constexpr int W_BYTES = WSMEM ? BM * RP * 2 : 0;   // one W tile in shared memory
  static constexpr int NWB = (RP == 256) ? 1 : 2;      // W tile buffers
  static constexpr int FREE = 512 - NWB * WCOLS - RCOLS;
  static constexpr int NB = FREE / BN >= 6 ? 6 : FREE / BN;  // L buffers
  static constexpr int PANEL_W = RP < 64 ? RP : 64;    // elements per row of one swizzle panel
  static constexpr int ROWB = PANEL_W * 2;             // bytes per panel row (= swizzle width)
  static constexpr int PANEL_BYTES = BN * ROWB;
  static constexpr int NPANEL = RP / PANEL_W;
  static constexpr int OPER_BYTES = BN * RP * 2;       // one bf16 piece of a chunk
  // bf16 pieces of each chunk in shared memory: hi in the bf16 mode, hi, lo
  // and lo2 in the fp32-accurate mode (hi and lo in its loss pass)
  static constexpr int NQ = SPLIT ? (LOSS ? 2 : 3) : 1;
  static constexpr int STAGE_BYTES = OPER_BYTES * NQ;
  // stages within 160 KB with the W tiles (r_pad <= 64: 165 KB in all, so
  // that an update block fits beside the CTA), 192 KB at r_pad = 128
  static constexpr int NSTAGE_RAW =
      ((WSMEM && RP <= 64) ? 160 * 1024 - NWB * W_BYTES : (WSMEM ? 192 * 1024 - NWB * W_BYTES : 160 * 1024)) /
      STAGE_BYTES;
  static constexpr int NSTAGE = NSTAGE_RAW > 8 ? 8 : (NSTAGE_RAW < 2 ? 2 : NSTAGE_RAW);
  static constexpr uint32_t SWZ = PANEL_W == 64 ? SWZ_128B : (PANEL_W == 32 ? SWZ_64B : SWZ_32B);
  // shared memory: stages, W tiles (WSMEM), barriers, TMEM slot + abort flag, ...
  static constexpr size_t OFF_W = (size_t)NSTAGE * STAGE_BYTES;
  static constexpr int W_PANEL_BYTES = BM * ROWB;     // one swizzle panel of a W tile
  static constexpr size_t OFF_BARS = OFF_W + (size_t)NWB * W_BYTES;
  static constexpr int COL_L = 0;               // NB x BN columns
  static constexpr int COL_R = NB * BN;         // RP columns
  static constexpr int COL_W = COL_R + RCOLS;   // NWB x WCOLS columns
  // barriers: full[NSTAGE], empty[NSTAGE], lfull[NB], pfull[NB], lfree[NB], rfull, rempty,
  // wfull[2], wempty[2], drain, drain2
  static constexpr int NBAR = 2 * NSTAGE + 3 * NB + 8;
  // after the barriers: TMEM slot and abort flag (64 B), the loss reduction
  // (256 x 16 B), and 4 flags per L buffer (Delta form: P nonzero per warp)
  static constexpr size_t SMEM_USED = 1024 + OFF_BARS + NBAR * 8 + 64 + 256 * 16 + NB * 16;
  // at least 120 KB so that a second CTA (and its 512-column TMEM request)
  // never shares the SM
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
  static_assert(NB >= 2, "need two L buffers");
  static_assert(NSTAGE >= 2, "stages");
  static_assert(SMEM <= 227 * 1024, "shared memory per block");
  static_assert(COL_W + NWB * WCOLS <= 512, "TMEM budget");
  static_assert(BN % 32 == 0 && RP % 16 == 0, "shapes");
};

struct TcParams {
  int64_t m0, M;        // M-side rows [m0, m0 + M) of the M factor
  int64_t q0, K;        // Q-side rows [q0, q0 + K) of the Q factor
  const bf16* Mhi;      // M factor operand copies (absolute row index)
  const bf16* Mlo;
  float* R;             // M x RP output (panel kernel)
  double* parts;        // per-CTA loss partials (loss kernel)
  int* status;
  float* Lout;          // verification: raw L (M x K, row-major) or nullptr
  const int64_t* rowptr;   // loss kernel: CSR of S, whose entries the dense pass skips
  const int32_t* cidx;
  unsigned long long* skips;   // Delta form: count of chunks whose second product was skipped (or nullptr)
  int skip_on;                 // Delta form: skip chunks whose rectified tile is zero
  // split K (steps with fewer tiles than SMs): CTA z takes Q-side rows
  // [q0 + z ksplit, ...) and writes its partial R at R + z rstride
  int64_t ksplit;              // 0: no split
  int64_t rstride;
  // range-search skipping (Delta form): bit c of tile t's words
  // rmask[t rwords ...] set = Q chunk c of the step is all L <= 0 for the
  // tile's rows (see range_mask_kernel); nullptr: no chunk is skipped
  const uint32_t* rmask;
  int64_t rwords;
  // nearest-neighbour pass (M side = Q side = one point set): per row the
  // largest L_ij over j != i, as an orderable key (value bits << 32 |
  // ~j); the caller zeroes the keys
  unsigned long long* nn_key;
  // update pass (M side = the step's right-hand side R, Q side = G^{-1}):
  // X = (R + Rs) G^{-1} with R and Rs fp32 rows (relative to the range, Rs
  // only where upd_flags is set) split into two bf16 pieces as they are
  // loaded; the epilogue applies the update of eqs. lsqA_sto / spLsqA to the
  // factor rows upd_row0 + i of upd_M (fp32 master), upd_E (momentum) and
  // upd_hi (bf16 piece)
  const float* upd_R;
  const float* upd_Rs;
  const uint8_t* upd_flags;
  float* upd_M;
  float* upd_E;
  bf16* upd_hi;
  int64_t upd_row0;
  float eta, gamma;
  int momentum, delta_form;
};

__device__ __forceinline__ void record(int* status, int code, int detail) {
  if (atomicCAS(status, 0, code) == 0) status[1] = detail;
}

// Bounded wait on an mbarrier phase.  Returns false if the kernel is aborting.
// The polls suspend in hardware until the phase completes (or 20 us pass), so
// waiting warps do not take issue slots from the MMA and copy threads.
__device__ __noinline__ bool wait_bar_slow(uint32_t bar, uint32_t parity, volatile int* abort_flag, int* status,
                                           int where, uint64_t limit_ns = kTimeoutNs) {
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) {
      *abort_flag = 1;
      record(status, NMD_ERR_TIMEOUT, where);
      return false;
    }
  }
}
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int* abort_flag, int* status,
                                         int where) {
  if (mbar_try_wait(bar, parity)) return true;
  return wait_bar_slow(bar, parity, abort_flag, status, where);
}

// Wait for a converged warp: every lane tests the phase; if it has not
// completed, lane 0 polls and the outcome is broadcast.
__device__ __forceinline__ bool conv_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, int* status,
                                          int where) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = wait_bar_slow(bar, parity, abort_flag, status, where);
  ok = __shfl_sync(0xffffffffu, ok, 0);
  return ok != 0;
}

// Warp-uniform wait: lane 0 polls, the outcome is broadcast to the warp.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, int* status,
                                          int where) {
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = wait_bar(bar, parity, abort_flag, status, where);
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

// The live Q chunks [0, n) of one tile (this CTA's split of it starts at
// chunk c0 of the tile's mask): those whose mask bit is clear.  A tile whose
// chunks are all masked still computes its chunk 0, which gives R = 0 (its L
// is <= 0 throughout), so that every tile has a first and a last chunk and
// the R hand-off is the same as without skipping.  The first 64 chunks'
// bits are kept in a register (a stochastic step has at most 64 chunks).
struct ChunkMask {
  const uint32_t* m;   // the tile's words, or nullptr (every chunk live)
  int64_t c0;
  bool none;           // every chunk masked
  uint64_t live64;     // bit c: chunk c (< 64) is live
  __device__ __forceinline__ bool masked_far(int64_t c) const {
    const int64_t b = c0 + c;
    return (m[b >> 5] >> (b & 31)) & 1u;
  }
  __device__ __forceinline__ bool live(int64_t c) const {
    if (m == nullptr) return true;
    if (none) return c == 0;
    return c < 64 ? ((live64 >> c) & 1ull) != 0 : !masked_far(c);
  }
};

template <bool RANGE>
__device__ __forceinline__ ChunkMask chunk_mask(const TcParams& p, int64_t t, int64_t c0, int64_t n,
                                                int64_t* last, int64_t* nlive) {
  ChunkMask cm{nullptr, c0, false, ~0ull};
  *last = n - 1;
  *nlive = n;
  if (!RANGE || p.rmask == nullptr) return cm;
  cm.m = p.rmask + t * p.rwords;
  // bits c0 .. c0 + 63 of the tile's words (words past the end read as masked)
  const int64_t w = c0 >> 5;
  const int sh = (int)(c0 & 31);
  const uint32_t w0 = w < p.rwords ? cm.m[w] : ~0u;
  const uint32_t w1 = w + 1 < p.rwords ? cm.m[w + 1] : ~0u;
  const uint32_t w2 = w + 2 < p.rwords ? cm.m[w + 2] : ~0u;
  const uint64_t lo = ((uint64_t)w1 << 32) | w0;
  const uint64_t bits = sh ? (lo >> sh) | ((uint64_t)w2 << (64 - sh)) : lo;
  const uint64_t inrange = n >= 64 ? ~0ull : ((1ull << n) - 1ull);
  cm.live64 = ~bits & inrange;
  int64_t cnt = __popcll(cm.live64), lst = cm.live64 ? 63 - __clzll(cm.live64) : -1;
  for (int64_t c = 64; c < n; ++c)
    if (!cm.masked_far(c)) {
      ++cnt;
      lst = c;
    }
  cm.none = cnt == 0;
  *last = cm.none ? 0 : lst;
  *nlive = cm.none ? 1 : cnt;
  return cm;
}

// MODE: 0 the panel contraction R = P(L) Q; 1 the loss pass (first product
// only, sums of max(0, L)^2 and max(0, L) off the support); 2 the nearest-
// neighbour pass (first product only, per row the largest L_ij, j != i);
// 3 the update pass (first product only: X = R G^{-1} and the step applied
// to the factor rows in the epilogue).
// SKIPM (Delta form only): 1 skips the second product of chunks whose
// rectified tile is zero (a vote of the epilogue warps); 2 skips both
// products of the chunks that the range-search mask clears.  Separate
// instantiations, so that the kernel without them carries none of the checks.
template <int RP, int EPI, bool SPLIT, int MODE, int SKIPM>
__global__ void __launch_bounds__(kThreads, 1)
    panel_tc_kernel(const __grid_constant__ CUtensorMap tq_hi, const __grid_constant__ CUtensorMap tq_lo,
                    const __grid_constant__ CUtensorMap tq_lo2, const __grid_constant__ CUtensorMap tw,
                    const TcParams p) {
  constexpr bool LOSS = MODE != 0;     // the first product only
  constexpr bool SUMS = MODE == 1, NEAREST = MODE == 2, UPDATE = MODE == 3;
  static_assert(!UPDATE || SPLIT, "the update pass splits R and G^{-1} into two pieces");
  // the update is skipped under a sticky error (as the CUDA-core update is);
  // every thread reads the same word before any barrier or TMEM exists
  if (UPDATE && *(volatile int*)p.status != 0) return;
  using C = Cfg<RP, SPLIT, LOSS>;
  constexpr int BN = C::BN, NB = C::NB, NSTAGE = C::NSTAGE, NWB = C::NWB;
  constexpr bool VOTE = SKIPM == 1, RANGE = SKIPM == 2;
  static_assert(SKIPM == 0 || (EPI == 1 && !LOSS), "skipping is a Delta-form option");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* stages = smem;
  const uint32_t wsm0 = smem_u32(smem + C::OFF_W);    // W tiles (WSMEM)
  uint64_t* bars = (uint64_t*)(smem + C::OFF_BARS);
  uint32_t* tmem_slot = (uint32_t*)(bars + C::NBAR);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);
  double* red = (double*)(smem + C::OFF_BARS + C::NBAR * 8 + 64);
  volatile uint32_t* pflag = (volatile uint32_t*)(red + 2 * kEpiThreads);   // [NB][4]

  const uint32_t b_full = smem_u32(bars);
  const uint32_t b_empty = b_full + 8 * NSTAGE;
  const uint32_t b_lfull = b_empty + 8 * NSTAGE;
  const uint32_t b_pfull = b_lfull + 8 * NB;
  const uint32_t b_lfree = b_pfull + 8 * NB;
  const uint32_t b_rfull = b_lfree + 8 * NB;
  const uint32_t b_rempty = b_rfull + 8;
  const uint32_t b_wfull = b_rempty + 8;
  const uint32_t b_wempty = b_wfull + 16;
  const uint32_t b_drain = b_wempty + 16;
  const uint32_t b_drain2 = b_drain + 8;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < NSTAGE; ++i) {
      mbar_init(b_full + 8 * i, 1);
      mbar_init(b_empty + 8 * i, 1);
    }
    for (int i = 0; i < NB; ++i) {
      mbar_init(b_lfull + 8 * i, 1);
      mbar_init(b_pfull + 8 * i, 4);                 // the four warps of one epilogue warpgroup
      mbar_init(b_lfree + 8 * i, LOSS ? 4 : 1);
    }
    mbar_init(b_rfull, 1);
    mbar_init(b_rempty, kEpiThreads / 32);
    for (int i = 0; i < 2; ++i) {
      mbar_init(b_wfull + 8 * i, C::WSMEM ? 1 : kEpiThreads / 32);   // TMA, or the epilogue warps
      mbar_init(b_wempty + 8 * i, 1);
    }
    mbar_init(b_drain, 1);
    mbar_init(b_drain2, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kProducerWarp) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
    if (lane == 0) {
      prefetch_tmap(&tq_hi);
      if (C::NQ > 1) prefetch_tmap(&tq_lo);
      if (C::NQ > 2) prefetch_tmap(&tq_lo2);
      if (C::WSMEM) prefetch_tmap(&tw);
    }
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = *tmem_slot;

  const int64_t ntiles = (p.M + BM - 1) / BM;
  const int64_t kz = blockIdx.z;
  const int64_t kq0 = p.ksplit ? p.q0 + kz * p.ksplit : p.q0;       // this CTA's Q-side rows
  const int64_t kK = p.ksplit ? (p.K - kz * p.ksplit < p.ksplit ? p.K - kz * p.ksplit : p.ksplit) : p.K;
  float* const Rout = p.ksplit ? p.R + kz * p.rstride : p.R;
  const int64_t nchunks = (kK + BN - 1) / BN;
  const int64_t kc0 = (kq0 - p.q0) / BN;   // this CTA's first chunk within the tile's mask

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int64_t G = 0, tt = 0;
      bool ok = true;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++tt) {
        if (C::WSMEM) {   // the tile's W rows into W buffer tt % NWB once MMA1 is done with it
          const int wb = (int)(tt % NWB);
          if (!(ok = wait_bar(b_wempty + 8 * wb, (uint32_t)((tt / NWB) & 1) ^ 1u, abort_flag, p.status, 10)))
            break;
          mbar_expect_tx(b_wfull + 8 * wb, C::W_BYTES);
#pragma unroll
          for (int pn = 0; pn < C::NPANEL; ++pn)
            tma_load_2d(wsm0 + wb * C::W_BYTES + pn * C::W_PANEL_BYTES, &tw, b_wfull + 8 * wb, pn * C::PANEL_W,
                        (int)(p.m0 + t * BM));
        }
        int64_t clast, nlive;
        const ChunkMask cm = chunk_mask<RANGE>(p, t, kc0, nchunks, &clast, &nlive);
        for (int64_t c = 0; c < nchunks; ++c) {
          if (RANGE && !cm.live(c)) continue;
          const int s = (int)(G % NSTAGE);
          if (!(ok = wait_bar(b_empty + 8 * s, (uint32_t)((G / NSTAGE) & 1) ^ 1u, abort_flag, p.status, 1)))
            break;
          mbar_expect_tx(b_full + 8 * s, C::STAGE_BYTES);
          const uint32_t dst = smem_u32(stages + (size_t)s * C::STAGE_BYTES);
          const int y = (int)(kq0 + c * BN);
#pragma unroll
          for (int pn = 0; pn < C::NPANEL; ++pn) {
            tma_load_2d(dst + pn * C::PANEL_BYTES, &tq_hi, b_full + 8 * s, pn * C::PANEL_W, y);
            if (C::NQ > 1)
              tma_load_2d(dst + C::OPER_BYTES + pn * C::PANEL_BYTES, &tq_lo, b_full + 8 * s, pn * C::PANEL_W, y);
            if (C::NQ > 2)
              tma_load_2d(dst + 2 * C::OPER_BYTES + pn * C::PANEL_BYTES, &tq_lo2, b_full + 8 * s, pn * C::PANEL_W,
                          y);
          }
          ++G;
        }
      }
      if (!ok) {  // drain the copies still in flight before shared memory goes away
        for (int64_t k = G - NSTAGE > 0 ? G - NSTAGE : 0; k < G; ++k) {
          uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(b_full + 8 * (int)(k % NSTAGE), (uint32_t)((k / NSTAGE) & 1)) &&
                 globaltimer_ns() - t0 < 100000000ull) {
          }
        }
        // W loads: those of tiles [0, tt) were issued, only the last NWB can
        // still be in flight
        for (int64_t k = tt - NWB > 0 ? tt - NWB : 0; C::WSMEM && k < tt; ++k) {
          uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(b_wfull + 8 * (int)(k % NWB), (uint32_t)((k / NWB) & 1)) &&
                 globaltimer_ns() - t0 < 100000000ull) {
          }
        }
      }
    }
  } else if (warp == kMma1Warp) {
    // ------------------------------------------------------------ MMA1 issuer
    // L[lb] = W tile x chunk^T for every chunk G of this CTA's tiles, in order.
    constexpr uint32_t idesc1 = idesc_bf16(BM, BN, false);   // Q K-major
    const uint32_t stage0 = smem_u32(stages);
    int s1 = 0, l1 = 0, wb1 = 0;
    uint32_t ph_full = 0, ph_lfree = 1, ph_wfull = 0;
    bool ok = true;
    for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
      int64_t clast, nlive;
      const ChunkMask cm = chunk_mask<RANGE>(p, t, kc0, nchunks, &clast, &nlive);
      if (RANGE && p.skips != nullptr && lane == 0 && nlive < nchunks)
        atomicAdd(p.skips, (unsigned long long)(nchunks - nlive));
      bool first = true;
      for (int64_t c = 0; c < nchunks; ++c) {
        if (RANGE && !cm.live(c)) continue;
        if (first && !(ok = conv_wait(b_wfull + 8 * wb1, ph_wfull, abort_flag, p.status, 2))) break;
        first = false;
        if (!(ok = conv_wait(b_full + 8 * s1, ph_full, abort_flag, p.status, 3))) break;
        if (!(ok = conv_wait(b_lfree + 8 * l1, ph_lfree, abort_flag, p.status, 4))) break;
        fence_after();
        const uint32_t wh = tmem + C::COL_W + wb1 * C::WCOLS;
        const uint32_t wl = wh + RP / 2;
        const uint64_t d1 = sdesc(stage0 + s1 * C::STAGE_BYTES, 16, 8 * C::ROWB, C::SWZ);
        // WSMEM: the W tile in the same K-major swizzled panels as a chunk
        const uint64_t a1 = sdesc(wsm0 + wb1 * C::W_BYTES, 16, 8 * C::ROWB, C::SWZ);
        const uint32_t d = tmem + C::COL_L + l1 * BN;
#pragma unroll
        for (int k = 0; k < RP / 16; ++k) {
          const uint32_t off = (k * 16 / C::PANEL_W) * C::PANEL_BYTES + ((k * 16) % C::PANEL_W) * 2;
          const uint64_t bh = d1 + (off >> 4);
          if (C::WSMEM)
            mma_ss_elect(d, a1 + (((k * 16 / C::PANEL_W) * C::W_PANEL_BYTES + ((k * 16) % C::PANEL_W) * 2) >> 4), bh,
                         idesc1, k > 0);
          else
            mma_ts_elect(d, wh + k * 8, bh, idesc1, k > 0);
          if (SPLIT) {
            const uint64_t bl = d1 + ((C::OPER_BYTES + off) >> 4);
            mma_ts_elect(d, wh + k * 8, bl, idesc1, 1);
            mma_ts_elect(d, wl + k * 8, bh, idesc1, 1);
          }
        }
        commit_elect(b_lfull + 8 * l1);
        if (LOSS) commit_elect(b_empty + 8 * s1);
        if (c == clast) commit_elect(b_wempty + 8 * wb1);
        if (++s1 == NSTAGE) { s1 = 0; ph_full ^= 1u; }
        if (++l1 == NB) { l1 = 0; ph_lfree ^= 1u; }
      }
      if (++wb1 == NWB) { wb1 = 0; ph_wfull ^= 1u; }
    }
    // wait until every MMA issued by this warp has completed
    commit_elect(b_drain);
    if (lane == 0) {
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(b_drain, 0) && globaltimer_ns() - t0 < 200000000ull) {
      }
    }
    __syncwarp();
  } else if (warp == kMma2Warp) {
    // ------------------------------------------------------------ MMA2 issuer
    // R += P[lb] x chunk for every chunk once its P is in TMEM; frees the
    // shared-memory stage and the L buffer, and hands R over per tile.
    if (!LOSS) {
      constexpr uint32_t idesc2 = idesc_bf16(BM, C::NR, true, EPI == 1 && !SPLIT);   // Q MN-major
      // R columns [hcol, hcol + NR) of Q: their panels start hcol / PANEL_W panels in
      const uint32_t hpan = C::RHALF ? (uint32_t)blockIdx.y * (C::NR / C::PANEL_W) * C::PANEL_BYTES : 0u;
      const uint32_t stage0 = smem_u32(stages);
      int s2 = 0, l2 = 0;
      uint32_t ph_pfull = 0, ph_rempty = 1;
      bool ok = true;
      for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        int64_t clast, nlive;
        const ChunkMask cm = chunk_mask<RANGE>(p, t, kc0, nchunks, &clast, &nlive);
        bool first = true;
        for (int64_t c = 0; c < nchunks; ++c) {
          if (RANGE && !cm.live(c)) continue;
          if (!(ok = conv_wait(b_pfull + 8 * l2, ph_pfull, abort_flag, p.status, 5))) break;
          if (first && !(ok = conv_wait(b_rempty, ph_rempty, abort_flag, p.status, 6))) break;
          fence_after();
          // Delta form: a chunk whose P is zero in every row adds nothing to R
          // (Sec. 4.3); its MMAs are skipped, except for the first chunk of a
          // tile, which initialises the accumulator
          bool skip = false;
          if (VOTE && !first)
            skip = (pflag[4 * l2] | pflag[4 * l2 + 1] | pflag[4 * l2 + 2] | pflag[4 * l2 + 3]) == 0u;
          if (VOTE && skip && p.skips != nullptr && lane == 0) atomicAdd(p.skips, 1ull);
          const uint64_t d2 = sdesc(stage0 + s2 * C::STAGE_BYTES + hpan, C::PANEL_BYTES, 8 * C::ROWB, C::SWZ);
          const uint32_t pl = tmem + C::COL_L + l2 * BN;
#pragma unroll
          for (int k = 0; k < BN / 16 && !(VOTE && skip); ++k) {
            const uint64_t bh = d2 + ((k * 16 * C::ROWB) >> 4);
            const uint32_t acc = (!first || k > 0) ? 1u : 0u;
            if (!SPLIT) {             // P q_hi
              mma_ts_elect(tmem + C::COL_R, pl + k * 8, bh, idesc2, acc);
            } else {                  // P_hi (q_hi + q_lo + q_lo2) + P_lo q_hi
              const uint64_t bl = bh + (C::OPER_BYTES >> 4);
              const uint64_t bl2 = bh + ((2 * C::OPER_BYTES) >> 4);
              const uint32_t ph = pl + (k / 2) * 32 + (k % 2) * 8, plo = ph + 16;
              mma_ts_elect(tmem + C::COL_R, ph, bh, idesc2, acc);
              mma_ts_elect(tmem + C::COL_R, ph, bl, idesc2, 1);
              mma_ts_elect(tmem + C::COL_R, ph, bl2, idesc2, 1);
              mma_ts_elect(tmem + C::COL_R, plo, bh, idesc2, 1);
            }
          }
          commit_elect(b_empty + 8 * s2);
          commit_elect(b_lfree + 8 * l2);
          if (c == clast) commit_elect(b_rfull);
          if (++s2 == NSTAGE) s2 = 0;
          if (++l2 == NB) { l2 = 0; ph_pfull ^= 1u; }
          if (first) ph_rempty ^= 1u;
          first = false;
        }
      }
      commit_elect(b_drain2);
      if (lane == 0) {
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(b_drain2, 0) && globaltimer_ns() - t0 < 200000000ull) {
        }
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // Two warpgroups take alternate chunks; within a warpgroup thread t owns
    // TMEM lane t = tile row t.  Tile-level work (W load, R readout) is split
    // by columns between the two warpgroups.
    const int wg = warp >> 2;
    const int row = (warp & 3) * 32 + lane;
    const int et = threadIdx.x;                          // 0 .. 255
    const uint32_t lane_base = ((uint32_t)((warp & 3) * 32)) << 16;
    double s2 = 0.0, s1 = 0.0;
    float nbest = -INFINITY;   // nearest-neighbour pass: this thread's best L of its row so far
    int64_t nidx = -1;
    bool ok = true;
    // loss pass: this thread's row of S, walked alongside the column chunks so
    // that support entries are left to the support pass (no cancellation)
    int64_t se = 0, send = 0;
    int64_t snext = INT64_MAX;

    // load the W tile `tile` into W buffer wb: warpgroup g takes 8-word groups g, g+2, ...
    auto load_w = [&](int64_t tile, int wb) {
      if constexpr (C::WSMEM) return;   // loaded by the producer's TMA
      const int64_t li = tile * BM + row;
      const bool valid = li < p.M;
      if constexpr (UPDATE) {
        // R + Rs of this row, split into hi = bf16(x) and lo = bf16(x - hi)
        const float* src = p.upd_R + (valid ? li : 0) * RP;
        const float* srs = p.upd_Rs + (valid ? li : 0) * RP;
        const bool flg = valid && p.upd_flags[li] != 0;
        const uint32_t wcol = tmem + lane_base + C::COL_W + wb * C::WCOLS;
#pragma unroll 1
        for (int q = wg; q < RP / 16; q += 2) {
          float x[16];
#pragma unroll
          for (int k = 0; k < 16; k += 4) {
            float4 a = valid ? __ldg((const float4*)(src + 16 * q + k)) : make_float4(0.f, 0.f, 0.f, 0.f);
            if (flg) {
              const float4 b = __ldg((const float4*)(srs + 16 * q + k));
              a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
            }
            x[k] = a.x; x[k + 1] = a.y; x[k + 2] = a.z; x[k + 3] = a.w;
          }
          uint32_t vh[8], vl[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t h = pack_bf16x2(x[2 * k], x[2 * k + 1]);
            vh[k] = h;
            vl[k] = pack_bf16x2(x[2 * k] - __uint_as_float(h << 16), x[2 * k + 1] - __uint_as_float(h & 0xffff0000u));
          }
          tmem_st8(wcol + q * 8, vh);
          tmem_st8(wcol + RP / 2 + q * 8, vl);
        }
        tmem_wait_st();
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(b_wfull + 8 * wb);
        return;
      }
      const uint4* src = (const uint4*)(p.Mhi + (p.m0 + (valid ? li : 0)) * RP);
      const uint4* srcl = (const uint4*)(p.Mlo + (p.m0 + (valid ? li : 0)) * RP);
      const uint32_t wcol = tmem + lane_base + C::COL_W + wb * C::WCOLS;
#pragma unroll
      for (int q = wg; q < RP / 16; q += 2) {
        uint4 a = valid ? __ldg(src + 2 * q) : make_uint4(0, 0, 0, 0);
        uint4 b = valid ? __ldg(src + 2 * q + 1) : make_uint4(0, 0, 0, 0);
        uint32_t v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        tmem_st8(wcol + q * 8, v);
        if (SPLIT) {
          uint4 c = valid ? __ldg(srcl + 2 * q) : make_uint4(0, 0, 0, 0);
          uint4 e = valid ? __ldg(srcl + 2 * q + 1) : make_uint4(0, 0, 0, 0);
          uint32_t w[8] = {c.x, c.y, c.z, c.w, e.x, e.y, e.z, e.w};
          tmem_st8(wcol + RP / 2 + q * 8, w);
        }
      }
      tmem_wait_st();
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_wfull + 8 * wb);
    };

    {  // prologue: the first NWB tiles
      int64_t tt = 0;
      for (int64_t t = blockIdx.x; t < ntiles && tt < NWB; t += gridDim.x, ++tt) load_w(t, (int)tt);
    }
    int64_t tt = 0;
    int64_t Gc = 0;   // chunks this CTA has processed
    for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++tt) {
      int64_t clast, nlive;
      const ChunkMask cm = chunk_mask<RANGE>(p, t, kc0, nchunks, &clast, &nlive);
      if (SUMS) {
        const int64_t li = t * BM + row;
        se = li < p.M ? p.rowptr[li] : 0;
        send = li < p.M ? p.rowptr[li + 1] : 0;
        snext = se < send ? p.cidx[se] : INT64_MAX;
      }
      for (int64_t c = 0; c < nchunks; ++c) {
        if (RANGE && !cm.live(c)) continue;
        const int64_t G = Gc++;
        if ((int)(G & 1) != wg) continue;
        if (SUMS) {   // skip the support columns of the other warpgroup's chunks
          while (snext < c * BN) {
            ++se;
            snext = se < send ? p.cidx[se] : INT64_MAX;
          }
        }
        const int lb = (int)(G % NB);
        if (!(ok = warp_wait(b_lfull + 8 * lb, (uint32_t)((G / NB) & 1), abort_flag, p.status, 7))) break;
        fence_after();
        const int kv = (int)(kK - c * BN < BN ? kK - c * BN : BN);   // valid columns in this chunk
        const uint32_t lcol = tmem + lane_base + C::COL_L + lb * BN;
        float c2 = 0.f, c1 = 0.f;
        uint32_t nzacc = 0u;   // Delta form: OR of this thread's P words
        // one group of 32 columns of L (TMEM columns [32 g, 32 g + 32) of the
        // buffer): mask the columns past the block, then the loss sums or P
        // (bf16, 16 TMEM columns at 16 g; fp32-accurate: hi and lo, 32 at 32 g,
        // so P never overwrites L columns that are still to be read)
        auto group = [&](uint32_t(&v)[32], int g) {
          if (kv < BN) {   // last chunk: columns past the block end contribute nothing
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (g * 32 + i >= kv) v[i] = SUMS ? 0u : (EPI == 0 ? 0u : 0xff800000u);   // -inf -> relu 0
          }
          if (p.Lout != nullptr) {
            const int64_t li = t * BM + row;
            if (li < p.M) {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (g * 32 + i < kv) p.Lout[li * p.K + c * BN + g * 32 + i] = __uint_as_float(v[i]);
            }
          }
          if (UPDATE) {   // X for columns [col0, col0 + 32) of this row: the step
            const int64_t li = t * BM + row;
            if (li < p.M) {
              const int64_t col0 = c * BN + g * 32;
              float* mrow = p.upd_M + (p.upd_row0 + li) * RP + col0;
              float* erow = p.upd_E + (p.upd_row0 + li) * RP + col0;
              uint32_t hw[16];
              bool finite = true;
#pragma unroll
              for (int k = 0; k < 32; k += 4) {
                const float4 mo = *(const float4*)(mrow + k);
                const float4 eo = p.momentum ? *(const float4*)(erow + k) : make_float4(0.f, 0.f, 0.f, 0.f);
                const float mv[4] = {mo.x, mo.y, mo.z, mo.w}, evo[4] = {eo.x, eo.y, eo.z, eo.w};
                float nv[4], ev[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                  const float x = __uint_as_float(v[k + j]);
                  const float u = p.delta_form ? p.eta * x : p.eta * (x - mv[j]);
                  ev[j] = p.momentum ? fmaf(p.gamma, evo[j], u) : u;
                  nv[j] = mv[j] + ev[j];
                  finite = finite && isfinite(nv[j]);
                }
                *(float4*)(mrow + k) = make_float4(nv[0], nv[1], nv[2], nv[3]);
                if (p.momentum) *(float4*)(erow + k) = make_float4(ev[0], ev[1], ev[2], ev[3]);
                hw[k / 2] = pack_bf16x2(nv[0], nv[1]);
                hw[k / 2 + 1] = pack_bf16x2(nv[2], nv[3]);
              }
              uint4* hrow = (uint4*)(p.upd_hi + (p.upd_row0 + li) * RP + col0);
#pragma unroll
              for (int k = 0; k < 4; ++k) hrow[k] = make_uint4(hw[4 * k], hw[4 * k + 1], hw[4 * k + 2], hw[4 * k + 3]);
              if (!finite) record(p.status, NMD_ERR_DIVERGED, (int)(p.upd_row0 + li));
            }
          } else if (NEAREST) {   // columns past the set or the row itself do not count
            const int64_t cb = c * BN + g * 32, self = t * BM + row;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float x = __uint_as_float(v[i]);
              if (g * 32 + i < kv && cb + i != self && x > nbest) {
                nbest = x;
                nidx = cb + i;
              }
            }
          } else if (SUMS) {
            const int64_t cb = c * BN + g * 32;
            if (snext < cb + 32) {   // support columns in this group: zero them
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                if (cb + i == snext) {
                  v[i] = 0u;
                  ++se;
                  snext = se < send ? p.cidx[se] : INT64_MAX;
                }
              }
            }
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              const float x0 = fmaxf(0.f, __uint_as_float(v[i])), x1 = fmaxf(0.f, __uint_as_float(v[i + 1]));
              c2 = fmaf(x0, x0, c2);
              c2 = fmaf(x1, x1, c2);
              c1 += x0 + x1;
            }
          } else if (!SPLIT) {
            uint32_t pk[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              if (EPI == 0) {   // min(0, L)
                pk[i] = min0_bf16x2(pack_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])));
              } else {          // max(0, L); the MMA negates it
                pk[i] = pack_relu_bf16x2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
                if (VOTE) nzacc |= pk[i] & 0x7fff7fffu;   // -0 counts as zero
              }
            }
            tmem_st16(lcol + g * 16, pk);
          } else {
            // fp32-accurate: P = hi + lo, hi at columns [32 g, 32 g + 16), lo at [32 g + 16, 32 g + 32)
            uint32_t ph[16], pl[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float x0 = __uint_as_float(v[2 * i]), x1 = __uint_as_float(v[2 * i + 1]);
              const float e0 = EPI == 0 ? fminf(0.f, x0) : fminf(0.f, -x0);
              const float e1 = EPI == 0 ? fminf(0.f, x1) : fminf(0.f, -x1);
              const uint32_t hp = pack_bf16x2(e0, e1);
              const float h0 = __uint_as_float(hp << 16), h1 = __uint_as_float(hp & 0xffff0000u);
              ph[i] = hp;
              pl[i] = pack_bf16x2(e0 - h0, e1 - h1);
              if (VOTE) nzacc |= (ph[i] | pl[i]) & 0x7fff7fffu;   // -0 counts as zero
            }
            tmem_st16(lcol + g * 32, ph);
            tmem_st16(lcol + g * 32 + 16, pl);
          }
        };
#pragma unroll 1
        for (int jj = 0; jj < BN / 64; ++jj) {   // two groups per pass, both loads in flight
          uint32_t v0[32], v1[32];
          tmem_ld32(lcol + jj * 64, v0);
          tmem_ld32(lcol + jj * 64 + 32, v1);
          tmem_wait_ld(v0);
          tmem_wait_ld(v1);
          group(v0, 2 * jj);
          group(v1, 2 * jj + 1);
        }
        if (BN % 64 != 0) {   // a last group of 32 columns
          uint32_t v0[32];
          tmem_ld32(lcol + (BN / 64) * 64, v0);
          tmem_wait_ld(v0);
          group(v0, BN / 32 - 1);
        }
        if (LOSS) {
          if (SUMS) {
            s2 += (double)c2;
            s1 += (double)c1;
          }
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_lfree + 8 * lb);
        } else {
          if (VOTE) {   // published before the arrive (release) that MMA2 acquires
            const bool nz = __any_sync(0xffffffffu, nzacc != 0u);
            if (lane == 0) pflag[4 * lb + (warp & 3)] = nz ? 1u : 0u;
          }
          tmem_wait_st();
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_pfull + 8 * lb);
        }
      }
      if (!ok) break;
      if (NEAREST) {   // this warpgroup's best of the row; the two are merged by atomicMax
        const int64_t li = t * BM + row;
        if (li < p.M && nidx >= 0) {
          const uint32_t b = __float_as_uint(nbest);
          const uint32_t ord = (b & 0x80000000u) ? ~b : (b | 0x80000000u);   // float order as unsigned
          atomicMax(p.nn_key + li, ((unsigned long long)ord << 32) | (unsigned long long)(~(uint32_t)nidx));
        }
        nbest = -INFINITY;
        nidx = -1;
      }
      if (!LOSS) {
        if (!(ok = warp_wait(b_rfull, (uint32_t)(tt & 1), abort_flag, p.status, 8))) break;
        fence_after();
        const int64_t li = t * BM + row;
        float* dst = Rout + li * RP + (C::RHALF ? (int64_t)blockIdx.y * C::NR : 0);
        constexpr int NJ = (C::NR + 31) / 32;
#pragma unroll 1
        for (int j = wg; j < NJ; j += 2) {
          // the warp's last TMEM read of the tile releases R (MMA2 may start
          // the next tile) before the adds and global stores
          const bool last = j + 2 >= NJ;
          uint32_t v[32];
          tmem_ld32(tmem + lane_base + C::COL_R + j * 32, v);   // RP = 16 reads 16 columns past R
          tmem_wait_ld(v);
          if (last) {
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(b_rempty);
          }
          if (li < p.M) {
#pragma unroll
            for (int i = 0; i < 32; i += 4)
              if (j * 32 + i < C::NR)
                *(float4*)(dst + j * 32 + i) = make_float4(__uint_as_float(v[i]), __uint_as_float(v[i + 1]),
                                                          __uint_as_float(v[i + 2]), __uint_as_float(v[i + 3]));
          }
        }
        if (wg >= NJ) {   // no columns for this warpgroup (r_pad = 16): release at once
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(b_rempty);
        }
      }
      // refill this tile's W buffer with the tile NWB steps ahead
      const int64_t tn = t + (int64_t)NWB * gridDim.x;
      if (!C::WSMEM && tn < ntiles) {
        const int wb = (int)(tt % NWB);
        if (!(ok = warp_wait(b_wempty + 8 * wb, (uint32_t)((tt / NWB) & 1), abort_flag, p.status, 9))) break;
        fence_after();
        load_w(tn, wb);
      }
    }
    if (SUMS) {
      // fixed-order reduction over the 256 epilogue threads
      red[2 * et] = s2;
      red[2 * et + 1] = s1;
      named_bar_sync(1, kEpiThreads);
      if (et == 0) {
        double a = 0.0, b = 0.0;
        for (int i = 0; i < kEpiThreads; ++i) {
          a += red[2 * i];
          b += red[2 * i + 1];
        }
        p.parts[(size_t)blockIdx.x * 8 + 0] = a;
        p.parts[(size_t)blockIdx.x * 8 + 1] = b;
      }
    }
  }
  fence_before();
  __syncthreads();
  fence_after();
  if (warp == kProducerWarp) tmem_dealloc(tmem, 512);
}

// Self-test of the bounded wait used by every pipeline wait above: thread 0
// waits on a barrier that nothing arrives at; after limit_ns the wait gives
// up, sets the abort flag and records NMD_ERR_TIMEOUT (detail 99) in the
// status words, and the kernel returns normally.
__global__ void wait_selftest_kernel(int* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) wait_bar_slow(smem_u32(&bar), 0, &abort_flag, status, 99, limit_ns);
  __syncthreads();
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
  });
  return fn;
}

// Tensor map of a row-major rows x rp bf16 factor copy, box = panel_w x bn.
bool tensor_map(const bf16* base, int64_t rows, int rp, int panel_w, int bn, CUtensorMap* out) {
  static std::mutex mu;
  static std::map<std::tuple<const void*, int64_t, int, int>, CUtensorMap> cache;
  std::lock_guard<std::mutex> g(mu);
  auto key = std::make_tuple((const void*)base, rows, rp, bn);
  auto it = cache.find(key);
  if (it != cache.end()) {
    *out = it->second;
    return true;
  }
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)rp, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)rp * 2};
  cuuint32_t box[2] = {(cuuint32_t)panel_w, (cuuint32_t)bn};
  cuuint32_t es[2] = {1, 1};
  CUtensorMapSwizzle swz = panel_w == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                         : (panel_w == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
  CUtensorMap m;
  CUresult r = fn(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)base, dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return false;
  cache[key] = m;
  *out = m;
  return true;
}

template <int RP, int EPI, bool SPLIT, int MODE, int SKIPM = 0>
nmd_status run(const Factor& fm, const Factor& fq, const TcParams& p, int grid, cudaStream_t s) {
  using C = Cfg<RP, SPLIT, MODE != 0>;
  CUtensorMap th, tl, tl2;
  if (!tensor_map(fq.hi, fq.rows, RP, C::PANEL_W, C::BN, &th)) return NMD_ERR_CUDA;
  if (!tensor_map(fq.lo, fq.rows, RP, C::PANEL_W, C::BN, &tl)) return NMD_ERR_CUDA;
  if (!tensor_map(fq.lo2, fq.rows, RP, C::PANEL_W, C::BN, &tl2)) return NMD_ERR_CUDA;
  // W tiles: the M-side rows [0, m0 + M) of the M factor's bf16 copy, so
  // that the rows of a ragged last tile past the block read as zero
  CUtensorMap tw = th;
  if (C::WSMEM && !tensor_map(fm.hi, p.m0 + p.M, RP, C::PANEL_W, BM, &tw)) return NMD_ERR_CUDA;
  // the shared-memory attributes belong to the current device.  At r_pad <=
  // 64 the carveout asks for the largest shared-memory configuration (228 KB
  // per SM): with the 166 KB of a CTA an SM would otherwise be set to 196 KB,
  // leaving no room for an update block (37 KB) beside it, and the deferred
  // update would run only on the SMs the grid leaves free.  (At r_pad = 256
  // the same setting slowed the sweep by 15%: there nothing fits beside a
  // CTA, and the L1 it takes away is lost.)
  static std::atomic<int> attr_set[kMaxDevices];
  if (!per_device(attr_set, [] {
        return (cudaFuncSetAttribute(panel_tc_kernel<RP, EPI, SPLIT, MODE, SKIPM>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM) == cudaSuccess &&
                (RP > 64 || cudaFuncSetAttribute(panel_tc_kernel<RP, EPI, SPLIT, MODE, SKIPM>,
                                                 cudaFuncAttributePreferredSharedMemoryCarveout,
                                                 100) == cudaSuccess)) ? 1 : 0;
      }))
    return NMD_ERR_CUDA;
  const unsigned gz = p.ksplit ? (unsigned)((p.K + p.ksplit - 1) / p.ksplit) : 1u;
  panel_tc_kernel<RP, EPI, SPLIT, MODE, SKIPM><<<dim3((unsigned)grid, C::RHALF ? 2u : 1u, gz), kThreads, C::SMEM, s>>>(
      th, tl, tl2, tw, p);
  return NMD_OK;
}

template <int RP, int MODE>
nmd_status dispatch_rp(int epilogue, bool split, const Factor& fm, const Factor& fq, const TcParams& p, int grid,
                       cudaStream_t s) {
  if constexpr (MODE == 2) {
    return run<RP, 0, true, 2>(fm, fq, p, grid, s);   // nearest neighbours: always the split pieces
  } else if constexpr (MODE == 1) {
    return split ? run<RP, 0, true, 1>(fm, fq, p, grid, s) : run<RP, 0, false, 1>(fm, fq, p, grid, s);
  }
  if (epilogue == NMD_EPI_DELTA && p.rmask != nullptr) {
    if (split) return run<RP, 1, true, 0, 2>(fm, fq, p, grid, s);
    return run<RP, 1, false, 0, 2>(fm, fq, p, grid, s);
  }
  if (epilogue == NMD_EPI_DELTA && p.skip_on) {
    if (split) return run<RP, 1, true, 0, 1>(fm, fq, p, grid, s);
    return run<RP, 1, false, 0, 1>(fm, fq, p, grid, s);
  }
  if (split)
    return epilogue == NMD_EPI_DELTA ? run<RP, 1, true, 0>(fm, fq, p, grid, s)
                                     : run<RP, 0, true, 0>(fm, fq, p, grid, s);
  return epilogue == NMD_EPI_DELTA ? run<RP, 1, false, 0>(fm, fq, p, grid, s)
                                   : run<RP, 0, false, 0>(fm, fq, p, grid, s);
}

template <int MODE>
nmd_status dispatch(int rp, int epilogue, bool split, const Factor& fm, const Factor& fq, const TcParams& p,
                    int grid, cudaStream_t s) {
  switch (rp) {
    case 16: return dispatch_rp<16, MODE>(epilogue, split, fm, fq, p, grid, s);
    case 32: return dispatch_rp<32, MODE>(epilogue, split, fm, fq, p, grid, s);
    case 64: return dispatch_rp<64, MODE>(epilogue, split, fm, fq, p, grid, s);
    case 128: return dispatch_rp<128, MODE>(epilogue, split, fm, fq, p, grid, s);
    case 256: return dispatch_rp<256, MODE>(epilogue, split, fm, fq, p, grid, s);
  }
  return NMD_ERR_UNSUPPORTED;
}

}  // namespace

int panel_chunk_rows(int rp, int precision) {
  const bool split = precision == NMD_FP32;
  switch (rp) {
    case 16: return split ? Cfg<16, true, false>::BN : Cfg<16, false, false>::BN;
    case 32: return split ? Cfg<32, true, false>::BN : Cfg<32, false, false>::BN;
    case 64: return split ? Cfg<64, true, false>::BN : Cfg<64, false, false>::BN;
    case 128: return split ? Cfg<128, true, false>::BN : Cfg<128, false, false>::BN;
    default: return split ? Cfg<256, true, false>::BN : Cfg<256, false, false>::BN;
  }
}

bool tc_supported(int rp, int precision) {
  if (precision == NMD_SIMT) return false;
  return rp == 16 || rp == 32 || rp == 64 || rp == 128 || rp == 256;
}

// R = sum over the splits of the partial R's, in split order
__global__ void split_reduce_kernel(const float* __restrict__ part, int64_t stride, int splits,
                                    float* __restrict__ R, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    float v = part[i];
    for (int z = 1; z < splits; ++z) v += part[z * stride + i];
    R[i] = v;
  }
}

nmd_status launch_panel_tc(const StepArgs& a, float* R, int* status, int* counter, int num_sms, cudaStream_t s,
                           int64_t* launches, float* Lout, float* rpart, int64_t rpart_rows) {
  if (!tc_supported(a.rp, a.precision)) return NMD_ERR_UNSUPPORTED;
  TcParams p{a.m0, a.M, a.q0, a.K, a.fm->hi, a.fm->lo, R, nullptr, status, Lout, nullptr, nullptr,
             (unsigned long long*)counter, a.skip_zero ? 1 : 0, 0, 0, a.rmask, a.rwords};
  const int64_t ntiles = (a.M + BM - 1) / BM;
  // a step with fewer tiles than SMs (the exact steps: b rows against all of
  // the other factor) splits K so that tiles x splits fill the SMs, each split
  // keeping at least 8 chunks; the partial R's are summed in split order
  int64_t splits = 1;
  if (Lout == nullptr && rpart != nullptr && ntiles < num_sms) {
    splits = std::min<int64_t>({(int64_t)num_sms / ntiles, (a.K + 64 * 8 - 1) / (64 * 8), 16,
                                rpart_rows / (ntiles * BM)});
    if (splits < 2) splits = 1;
  }
  int grid;
  if (splits > 1) {
    p.ksplit = ((a.K + splits - 1) / splits + 127) / 128 * 128;   // whole chunks of 64 or 128 rows
    splits = (a.K + p.ksplit - 1) / p.ksplit;
    p.R = rpart;
    p.rstride = a.M * a.rp;
    grid = (int)ntiles;
  } else {
    // fewest CTAs that keep the same number of tile rounds: the SMs left over
    // run the side-stream kernels of the step
    const int64_t rounds = (ntiles + num_sms - 1) / num_sms;
    grid = (int)((ntiles + rounds - 1) / rounds);
  }
  nmd_status st = dispatch<0>(a.rp, a.epilogue, a.precision == NMD_FP32, *a.fm, *a.fq, p, grid, s);
  if (st != NMD_OK) return st;
  ++*launches;
  if (splits > 1) {
    const int64_t n = a.M * a.rp;
    const int64_t blocks = std::min<int64_t>((n + 255) / 256, (int64_t)num_sms * 8);
    split_reduce_kernel<<<(unsigned)blocks, 256, 0, s>>>(rpart, p.rstride, (int)splits, R, n);
    ++*launches;
  }
  return NMD_OK;
}

void launch_wait_selftest(int* status, uint64_t limit_ns, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(status, limit_ns);
}

nmd_status launch_update_tc(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags,
                            const Factor& gi, float eta, float gamma, bool momentum, int* status, int num_sms,
                            cudaStream_t s) {
  if (a.M <= 0) return NMD_OK;
  TcParams p{0, a.M, 0, a.rp, nullptr, nullptr, nullptr, nullptr, status, nullptr, nullptr, nullptr, nullptr, 0,
             0, 0, nullptr, 0, nullptr, R, Rs, flags, a.fm->master, a.fm->E, a.fm->hi, a.m0, eta, gamma,
             momentum ? 1 : 0, a.epilogue == NMD_EPI_DELTA ? 1 : 0};
  const int64_t ntiles = (a.M + BM - 1) / BM;
  const int64_t rounds = (ntiles + num_sms - 1) / num_sms;
  const int grid = (int)((ntiles + rounds - 1) / rounds);
  if (a.rp != 256) return NMD_ERR_UNSUPPORTED;
  return run<256, 0, true, 3>(*a.fm, gi, p, grid, s);
}

nmd_status launch_nearest_tc(const Factor& f, int64_t N, int rp, unsigned long long* keys, int* status,
                             int num_sms, cudaStream_t s) {
  if (!tc_supported(rp, NMD_FP32)) return NMD_ERR_UNSUPPORTED;
  TcParams p{0, N, 0, N, f.hi, f.lo, nullptr, nullptr, status, nullptr, nullptr, nullptr, nullptr, 0, 0, 0,
             nullptr, 0, keys};
  const int64_t ntiles = (N + BM - 1) / BM;
  const int64_t rounds = (ntiles + num_sms - 1) / num_sms;
  const int grid = (int)((ntiles + rounds - 1) / rounds);
  return dispatch<2>(rp, 0, true, f, f, p, grid, s);
}

nmd_status launch_loss_dense_tc(const nmd_handle* h, double* parts, int maxparts, int* nparts, int* status,
                                cudaStream_t s, int64_t* launches) {
  if (!tc_supported(h->rp, h->opt.precision)) return NMD_ERR_UNSUPPORTED;
  TcParams p{0, h->m, 0, h->n, h->W.hi, h->W.lo, nullptr, parts, status, nullptr, h->ws.rowptr, h->ws.col,
             nullptr, 0, 0, 0};
  int64_t ntiles = (h->m + BM - 1) / BM;
  int grid = (int)(ntiles < h->num_sms ? ntiles : h->num_sms);
  if (grid > maxparts) grid = maxparts;
  nmd_status st = dispatch<1>(h->rp, 0, h->opt.precision == NMD_FP32, h->W, h->B, p, grid, s);
  if (st == NMD_OK) {
    ++*launches;
    *nparts = grid;
  }
  return st;
}

}  // namespace nmd
