// Fused LR-QAT GEMM for the forward (Y = X W_hat^T) and the input gradient
// (dX = dY W_hat) on CTA pairs: the same on-chip recompute of W_hat as the one-SM
// kernel (Eq. 8; the recompute replaces the checkpointing of Sec. 3), with the main
// product issued as tcgen05 MMAs of M = 256 rows across the two SMs of a cluster.
//
// Why pairs: the one-SM kernel (128 x 448 tiles) moves its whole 448-token operand through
// each SM's shared memory every stage; in a pair each CTA holds its own 128 weight rows and only
// half of every accumulator's tokens, and the tensor cores of the pair exchange the token halves
// (measured on a 4096 x 4096 layer at T = 8192 on the codes: forward 276 -> 181 us).
//
// A pair processes tiles of 256 weight rows (CTA rank c: rows 128 c .. 128 c + 127) x 448
// tokens (two accumulators of 224 tokens; CTA c holds tokens 112 c .. 112 c + 111 of each), one
// 64-wide slice of the contraction per stage:
//   * token ring (three slots per CTA, four on the codes): one loader warp per slot brings this
//     CTA's two 112-token halves (SW128) with TMA whose completion lands on the leader's
//     barrier; each slot also holds this CTA's W_hat tile of the stage;
//   * factor ring (4 slots; 2 for 16-bit bases): the stored base of this CTA's rows (completion
//     on its own barrier; only its own producers read it), with it the stage's scales (and zero
//     offsets) where the producers apply them (dX, group-wise forward), and with the low-rank tile
//     this CTA's half (32 rows) of the second factor's slice (completion on the leader's
//     barrier: the low-rank MMA reads both halves);
//   * in the leader, one thread issues the main product (M = 256, N = 224, 8 MMAs per stage) and,
//     with the low-rank tile in the stage, another the tile L = RF SF^T (M = 256, N = 64) into a
//     TMEM buffer after the accumulators, so that neither waits behind the other's barriers;
//     every commit is multicast to both CTAs;
//   * sixteen producer warps per CTA build this CTA's W_hat tile exactly as the one-SM kernel
//     does (on the codes, two stages per iteration), and drain this CTA's 128 rows of the
//     accumulators in the epilogue.
// One barrier per slot in the leader counts the stage's token bytes and both CTAs' "W_hat
// written" events, so the MMA thread tests one barrier per stage; the peer's events ("W_hat
// written", "L read", "accumulators drained") travel as 16-byte copies into the leader's shared
// memory whose completion counts on the leader's barrier (a thread-issued remote arrive is
// several times slower under the pair's operand traffic), after fence.proxy.async has ordered
// the peer's writes.
// On the codes (NL: every rank from 3072 tokens on, and ranks above 64) the base holds the
// one-byte codes of the codes pass; no factors, no L.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int BM = 128;                          // weight rows per CTA (256 per pair)
constexpr int BK = 64;
constexpr int BNP = 224;                         // tokens per accumulator (N of the pair MMA)
constexpr int BNH = BNP / 2;                     // tokens per accumulator held by one CTA
constexpr int NACC = 2;
constexpr int BTP = BNP * NACC;                  // 448 tokens per pair tile
constexpr int NT_MAX = 4;                        // token ring slots (3 with the low-rank tile)
constexpr int NLB = 1;                           // low-rank TMEM buffers
constexpr int NF_MAX = 4;                        // factor ring slots (2 for 16-bit bases)
constexpr int NUM_PROD_WARPS = 16;
constexpr int FIRST_TMA_WARP = 2 + NUM_PROD_WARPS;
constexpr int NUM_TMA_WARPS = NT_MAX + 1;        // a token loader per slot, the factor loader
constexpr int NUM_THREADS = 32 * (FIRST_TMA_WARP + NUM_TMA_WARPS);
constexpr int EPI_COLS = NACC * BNP / 4;         // accumulator columns drained per warp (112)
constexpr uint32_t SIG_TX = 16u * NUM_PROD_WARPS;   // bytes of the peer's per-warp signals

constexpr uint32_t RF_BYTES = 128 * 128;         // 128 rows x 64 rank columns (bf16)
constexpr uint32_t TOK_BOX = BNH * 128;          // 112 tokens x 64 bf16
constexpr uint32_t TOK_BYTES = NACC * TOK_BOX;
constexpr uint32_t W_BYTES = 128 * 128;          // 128 rows x 64 bf16
constexpr uint32_t SFH_BYTES = 32 * 128;         // 32 slice rows x up to 64 rank columns (bf16)
constexpr uint32_t TSLOT_BYTES = TOK_BYTES + W_BYTES;
constexpr uint32_t TS_W = TOK_BYTES;

// Shared-memory rings.  With the low-rank tile: the row factor, three token slots and per stage
// the stored base and this CTA's half of the second factor's slice.  On the codes (NL): no
// factors, so a fourth token slot fits (measured on a 4096 x 4096 layer at T = 8192: forward
// 191 -> 181 us).
// XS: each factor slot also holds the stage's scales (and zero offsets) as bf16, copied by the
// factor loader, so that the producers read them from shared memory with the base instead of
// from global memory: for dX the 64 scales of the stage's contraction indices in the CTA's row
// group, for the group-wise forward the 128 scales of the CTA's rows in the stage's group.
template <int FMT, bool NL, bool XS>
struct PairRing {
  static constexpr int NT = NL ? 4 : 3;
  static constexpr int NF = fmt_16bit(FMT) ? 2 : 4;
  static constexpr uint32_t RF = NL ? 0u : RF_BYTES;
  static constexpr uint32_t PHI_BYTES = fmt_16bit(FMT) ? 128 * 128 : 128 * 64;
  static constexpr uint32_t PHI_TX = FMT == FMT_I4 ? PHI_BYTES / 2 : PHI_BYTES;
  static constexpr uint32_t FS_SF = PHI_BYTES;
  // scales at +0, zero offsets at +512 (dX: 128 bytes each, group-wise forward: 256)
  static constexpr uint32_t FS_X = PHI_BYTES + (NL ? 0u : SFH_BYTES);
  static constexpr uint32_t FSLOT_BYTES = FS_X + (XS ? 1024u : 0u);
  static constexpr uint32_t OFF_RF = 0;
  static constexpr uint32_t OFF_TSLOTS = RF;
  static constexpr uint32_t OFF_FSLOTS = OFF_TSLOTS + NT * TSLOT_BYTES;
  static constexpr uint32_t SMEM_BYTES = OFF_FSLOTS + NF * FSLOT_BYTES + 1024;
  static_assert(NT <= NT_MAX, "token slots");
  static_assert(FSLOT_BYTES % 1024 == 0 && FS_SF % 1024 == 0 && OFF_FSLOTS % 1024 == 0,
                "swizzled tiles must start on 1024-byte boundaries");
  static_assert(SMEM_BYTES + 1024 <= 232448, "shared memory budget");
};
static_assert(TSLOT_BYTES % 1024 == 0 && TOK_BOX % 1024 == 0 && TS_W % 1024 == 0,
              "swizzled tiles must start on 1024-byte boundaries");
static_assert(EPI_COLS % 16 == 0, "epilogue drains 16-column chunks");

constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_L = NACC * BNP;           // the 64-column low-rank buffer(s) after the accumulators
static_assert(COL_L + NLB * BK <= TMEM_COLS, "TMEM budget");

// leader: the stage's operands are in place, i.e. both token halves of the slot landed and both
// CTAs' producers wrote their W_hat tiles (one barrier, so that the MMA thread tests one per stage)
constexpr int BAR_TFULL = 0;
constexpr int BAR_TEMPTY = BAR_TFULL + NT_MAX;   // both: main product of the slot finished
constexpr int BAR_PFULL = BAR_TEMPTY + NT_MAX;   // both: this CTA's base tile landed

constexpr int BAR_FFULL = BAR_PFULL + NF_MAX;    // leader: both factor-slice halves landed
constexpr int BAR_FEMPTY = BAR_FFULL + NF_MAX;   // both: slot read by this CTA's producers (after L)
constexpr int BAR_LFULL = BAR_FEMPTY + NF_MAX;   // both: low-rank tile of the buffer computed
constexpr int BAR_LEMPTY = BAR_LFULL + NLB;      // leader: both CTAs read the buffer
constexpr int BAR_RFFULL = BAR_LEMPTY + NLB;     // leader: both row-factor halves landed
constexpr int BAR_RFEMPTY = BAR_RFFULL + 1;      // both: last low-rank MMA of the tile finished
constexpr int BAR_ACCFULL = BAR_RFEMPTY + 1;     // both: accumulators of the tile complete
constexpr int BAR_ACCEMPTY = BAR_ACCFULL + 1;    // leader: both CTAs drained them
constexpr int BAR_DRAIN = BAR_ACCEMPTY + 1;
constexpr int NUM_BARS = BAR_DRAIN + 1;

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) break;
  }
}

// Stages are numbered globally over the pair's tiles (gg), identically in both CTAs: token
// slot gg % NT, factor slot gg % NF, low-rank buffer gg % 2.
template <int MODE, int FMT, bool ZP, bool UB, bool NL>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    fused_pair_kernel(const __grid_constant__ CUtensorMap tm_tok, const __grid_constant__ CUtensorMap tm_phi,
                      const __grid_constant__ CUtensorMap tm_rf, const __grid_constant__ CUtensorMap tm_sf,
                      const FusedArgs args) {
  using PR = PairRing<FMT, NL, MODE == FUSED_DX || MODE == FUSED_FWD_GROUP>;
  constexpr int NT = PR::NT;
  constexpr int NF = PR::NF;
  constexpr uint32_t OFF_RF = PR::OFF_RF, OFF_TSLOTS = PR::OFF_TSLOTS, OFF_FSLOTS = PR::OFF_FSLOTS;
  constexpr bool PACKED = FMT == FMT_I4;
  constexpr uint32_t FSLOT_BYTES = PR::FSLOT_BYTES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[NUM_BARS];
  __shared__ __align__(16) uint32_t sig_buf[8];   // [0, 4): source of the peer's signals, [4, 8): their target
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int abort_s;

  const uint32_t smem = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_cta_rank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  auto lbar = [&](int i) { return map_shared_rank(smem_u32(&bars[i]), 0); };   // the leader's copy

  if (threadIdx.x == 0) {
    abort_s = 0;
    for (int s = 0; s < NT; ++s) {
      mbar_init(bar(BAR_TFULL + s), 1 + NUM_PROD_WARPS);   // the leader's token loader and producer warps
      mbar_init(bar(BAR_TEMPTY + s), 1);
    }
    for (int s = 0; s < NF; ++s) {
      mbar_init(bar(BAR_PFULL + s), 1);
      mbar_init(bar(BAR_FFULL + s), 1);
      // freed by this CTA's producers after they built W_hat: by then they have waited for the
      // low-rank tile, so the low-rank MMA that read the slot's factor half has completed
      mbar_init(bar(BAR_FEMPTY + s), NUM_PROD_WARPS);
    }
    for (int b = 0; b < NLB; ++b) {
      mbar_init(bar(BAR_LFULL + b), 1);
      mbar_init(bar(BAR_LEMPTY + b), NUM_PROD_WARPS);
    }
    mbar_init(bar(BAR_RFFULL), 1);
    mbar_init(bar(BAR_RFEMPTY), 1);
    mbar_init(bar(BAR_ACCFULL), 1);
    mbar_init(bar(BAR_ACCEMPTY), NUM_PROD_WARPS);
    mbar_init(bar(BAR_DRAIN), 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc_pair(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};
  const int nk = args.kdim / BK;   // at least 2 (kdim is a multiple of 128)
  const int num_rb2 = args.num_rb / 2;   // 256-row blocks
  const int num_tiles = num_rb2 * ((args.T + BTP - 1) / BTP);
  const uint32_t sig_src = smem_u32(&sig_buf[0]);
  const uint32_t sig_dst_leader = map_shared_rank(smem_u32(&sig_buf[4]), 0);
  // A producer warp's event on a leader barrier: the leader's warps arrive (warp 0 also
  // announces the peer's 16 signal bytes per warp), the peer's warps send their signal.
  auto report = [&](int b, int pw) {
    if (leader) {
      if (pw == 0) mbar_arrive_expect_tx(bar(b), SIG_TX);
      else mbar_arrive(bar(b));
    } else {
      signal_remote16(sig_dst_leader, sig_src, lbar(b));
    }
  };

  if (warp == 0) {
    // ------------------- row factor (per tile) and, in the leader, the low-rank MMAs
    // A thread of its own issues the low-rank tiles, so that the main product never waits
    // behind their barriers; each thread's commits track only its own MMAs.
    if (!NL && lane == 0) {
      prefetch_tensormap(&tm_rf);
      const uint32_t idesc_l = make_idesc_bf16(256, BK, 0, 0);
      const int lsteps = args.r16 / 16;
      const uint64_t d_rf = make_sdesc(smem + OFF_RF, 16, 1024, SWZ_128B);
      // the K-major half slice: 32 rows of sf_cols bf16 (32, 64 or 128 bytes, swizzled to match)
      const uint32_t sf_swz = args.sf_cols == 64 ? SWZ_128B : args.sf_cols == 32 ? SWZ_64B : SWZ_32B;
      const uint64_t d_sf0 = make_sdesc(smem + OFF_FSLOTS + PR::FS_SF, 16, 16u * args.sf_cols, sf_swz);
      constexpr uint32_t FSLOT_D = FSLOT_BYTES >> 4;
      uint32_t it = 0, g = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
        const int rb2 = tile % num_rb2;
        if (!(ok = wait_spin_bounded(bar(BAR_RFEMPTY), (it & 1u) ^ 1u, ctl, 1))) break;
        if (leader) mbar_arrive_expect_tx(bar(BAR_RFFULL), 2u * RF_BYTES);
        tma_load_2d_pair(smem + OFF_RF, &tm_rf, 0, rb2 * 2 * BM + static_cast<int>(rank) * BM, lbar(BAR_RFFULL));
        if (leader) {
          if (!(ok = wait_spin_bounded(bar(BAR_RFFULL), it & 1u, ctl, 6))) break;
          for (int kk = 0; kk < nk && ok; ++kk) {
            // L(gg) into buffer gg % NLB once both factor halves landed and both CTAs read L(gg - NLB)
            const uint32_t gg = g + kk, s = gg % NF, b = gg % NLB;
            if (!(ok = wait_spin_bounded(bar(BAR_FFULL + s), (gg / NF) & 1u, ctl, 4))) break;
            if (!(ok = wait_spin_bounded(bar(BAR_LEMPTY + b), ((gg / NLB) & 1u) ^ 1u, ctl, 5))) break;
            tc_fence_after();
            const uint64_t sf = d_sf0 + s * FSLOT_D;
            const uint32_t dl = tmem + COL_L + BK * b;
            for (int ks = 0; ks < lsteps; ++ks) mma_bf16_pair(dl, d_rf + 2 * ks, sf + 2 * ks, idesc_l, ks > 0 ? 1u : 0u);
            mma_commit_pair(bar(BAR_LFULL + b));
          }
          if (!ok) break;
          mma_commit_pair(bar(BAR_RFEMPTY));   // last read of the row factor issued
        }
        g += nk;
        ++it;
      }
      if (leader && ok) {
        // the peer's reports of the last low-rank tiles land before the CTAs end
        for (uint32_t gg = g >= NLB ? g - NLB : 0; ok && gg < g; ++gg)
          ok = wait_spin_bounded(bar(BAR_LEMPTY + gg % NLB), (gg / NLB) & 1u, ctl, 11);
      }
    }
  } else if (warp >= FIRST_TMA_WARP && warp < FIRST_TMA_WARP + NT_MAX) {
    // ------------------------------------------- token loaders (one per slot)
    const uint32_t t = warp - FIRST_TMA_WARP;   // slots past NT have no loader work
    if (lane == 0 && t < static_cast<uint32_t>(NT)) {
      prefetch_tensormap(&tm_tok);
      const uint32_t st = smem + OFF_TSLOTS + t * TSLOT_BYTES;
      const uint32_t fb = lbar(BAR_TFULL + t), eb = bar(BAR_TEMPTY + t);
      uint32_t g = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
        const int tb = tile / num_rb2;
        for (int kk = 0; kk < nk; ++kk) {
          const uint32_t gg = g + kk;
          if (gg % NT != t) continue;
          const uint32_t n = gg / NT;
          if (!(ok = wait_spin_bounded(eb, (n & 1u) ^ 1u, ctl, 2))) break;
          if (leader) mbar_arrive_expect_tx(bar(BAR_TFULL + t), 2u * TOK_BYTES);
          const int tok = tb * BTP + static_cast<int>(rank) * BNH;
          tma_load_2d_pair(st, &tm_tok, kk * BK, tok, fb);
          tma_load_2d_pair(st + TOK_BOX, &tm_tok, kk * BK, tok + BNP, fb);
        }
        g += nk;
      }
    }
  } else if (warp == FIRST_TMA_WARP + NT_MAX) {
    // ------------------------------------------------- factor-ring loader
    if (lane == 0) {
      prefetch_tensormap(&tm_phi);
      if (!NL) prefetch_tensormap(&tm_sf);
      const uint32_t sf_tx = static_cast<uint32_t>(32 * 2 * args.sf_cols);   // one CTA's half slice
      uint32_t gg = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
        const int rb2 = tile % num_rb2;
        for (int kk = 0; kk < nk; ++kk, ++gg) {
          const uint32_t s = gg % NF;
          if (!(ok = wait_spin_bounded(bar(BAR_FEMPTY + s), ((gg / NF) & 1u) ^ 1u, ctl, 3))) break;
          const uint32_t fs = smem + OFF_FSLOTS + s * FSLOT_BYTES;
          constexpr uint32_t XTX = MODE == FUSED_DX        ? (ZP ? 256u : 128u)
                                   : MODE == FUSED_FWD_GROUP ? (ZP ? 512u : 256u)
                                                             : 0u;
          mbar_arrive_expect_tx(bar(BAR_PFULL + s), PR::PHI_TX + XTX);
          tma_load_2d(fs, &tm_phi, PACKED ? kk * (BK / 2) : kk * BK, rb2 * 2 * BM + static_cast<int>(rank) * BM,
                      bar(BAR_PFULL + s));
          if (MODE == FUSED_DX) {
            // the stage's 64 scales (and zero offsets) of this CTA's row group (group sizes are
            // multiples of 128, so a CTA's 128 rows lie in one group)
            const int64_t xoff = (args.s_ld ? static_cast<int64_t>((rb2 * 2 * BM + static_cast<int>(rank) * BM) /
                                                                   args.group_size) * args.kdim
                                            : 0) + kk * BK;
            bulk_load(fs + PR::FS_X, args.s_bf16 + xoff, 128u, bar(BAR_PFULL + s));
            if (ZP) bulk_load(fs + PR::FS_X + 512u, args.z_bf16 + xoff, 128u, bar(BAR_PFULL + s));
          } else if (MODE == FUSED_FWD_GROUP) {
            // the 128 scales (and zero offsets) of this CTA's rows in the stage's group, from the
            // bf16 rows [groups][m] (a group holds a multiple of 128 contraction indices, so two
            // stages never straddle it)
            const int64_t xoff = static_cast<int64_t>((kk * BK) / args.group_size) * args.rows + rb2 * 2 * BM +
                                 static_cast<int>(rank) * BM;
            bulk_load(fs + PR::FS_X, args.s_bf16 + xoff, 256u, bar(BAR_PFULL + s));
            if (ZP) bulk_load(fs + PR::FS_X + 512u, args.z_bf16 + xoff, 256u, bar(BAR_PFULL + s));
          }
          if (!NL) {
            if (leader) mbar_arrive_expect_tx(bar(BAR_FFULL + s), 2u * sf_tx);
            tma_load_2d_pair(fs + PR::FS_SF, &tm_sf, 0, kk * BK + static_cast<int>(rank) * 32, lbar(BAR_FFULL + s));
          }
        }
      }
      if (gg > 0) {
        const uint32_t last = gg - 1;
        drain_wait(bar(BAR_PFULL + last % NF), (last / NF) & 1u, args.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------ main-product MMA issuer (the leader's)
    if (leader && lane == 0) {
      const uint32_t idesc_main = make_idesc_bf16(256, BNP, 0, 0);
      constexpr uint32_t TSLOT_D = TSLOT_BYTES >> 4, TOKB_D = TOK_BOX >> 4;
      const uint64_t d_w0 = make_sdesc(smem + OFF_TSLOTS + TS_W, 16, 1024, SWZ_128B);
      const uint64_t d_tok0 = make_sdesc(smem + OFF_TSLOTS, 16, 1024, SWZ_128B);
      uint32_t g = 0, it = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
        if (!(ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 7))) break;
        tc_fence_after();
        // unrolled: the loop's own overhead between two stages' MMAs was ~120 cycles of idle tensor pipe
#pragma unroll 4
        for (int kk = 0; kk < nk; ++kk) {
          const uint32_t gg = g + kk;
          const uint32_t s = gg % NT, ph = (gg / NT) & 1u;
          if (!(ok = wait_spin_bounded(bar(BAR_TFULL + s), ph, ctl, 9))) break;
          tc_fence_after();
          const uint64_t w = d_w0 + s * TSLOT_D, t = d_tok0 + s * TSLOT_D;
          const uint32_t acc = kk > 0 ? 1u : 0u;
          static_assert(NACC == 2 && BK == 64, "issue sequence below is written for 2 accumulators x 4 K steps");
          mma_bf16_pair(tmem, w, t, idesc_main, acc);
          mma_bf16_pair(tmem, w + 2, t + 2, idesc_main, 1u);
          mma_bf16_pair(tmem, w + 4, t + 4, idesc_main, 1u);
          mma_bf16_pair(tmem, w + 6, t + 6, idesc_main, 1u);
          mma_bf16_pair(tmem + BNP, w, t + TOKB_D, idesc_main, acc);
          mma_bf16_pair(tmem + BNP, w + 2, t + TOKB_D + 2, idesc_main, 1u);
          mma_bf16_pair(tmem + BNP, w + 4, t + TOKB_D + 4, idesc_main, 1u);
          mma_bf16_pair(tmem + BNP, w + 6, t + TOKB_D + 6, idesc_main, 1u);
          mma_commit_pair(bar(BAR_TEMPTY + s));
        }
        if (!ok) break;
        mma_commit_pair(bar(BAR_ACCFULL));
        g += nk;
        ++it;
      }
      // the peer's last drain report lands before the CTAs end
      if (ok) ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 10);
      mma_commit_pair_self(bar(BAR_DRAIN));
      drain_wait(bar(BAR_DRAIN), 0, args.timeout_ns);
    }
  } else {
    // ------------------------------------------- W_hat producers + epilogue
    const int pw = warp - 2;              // 0..15
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int c = pw >> 2;                // 16-column chunk of the 64-wide slice (and epilogue block)
    const int row = q * 32 + lane;        // row of this CTA's tile handled by this thread
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const QuantParams qp = args.q;
    const uint32_t lr2 = pack_rn_bf16x2(qp.lr_scale, qp.lr_scale);
    // On the codes each warp builds two stages per iteration: both bases are read before either is
    // decoded and one proxy fence covers both W_hat stores, so that the per-stage chain of
    // shared-memory round trips (base read, W_hat store, fence, reports) is paid once per two
    // stages (kdim is a multiple of 128, so nk is even).
    constexpr int SPI = NL ? 2 : 1;
    uint32_t g = 0;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = pair; tile < num_tiles && ok; tile += npairs) {
      const int rb2 = tile % num_rb2;
      const int tb = tile / num_rb2;
      const int row_g = rb2 * 2 * BM + static_cast<int>(rank) * BM + row;
      for (int kk = 0; kk < nk; kk += SPI) {
        uint32_t scw[SPI][8];   // dX: the stage's 16 bf16 scales of its contraction indices, as bf16x2
        uint32_t zw[SPI][8];    // zero offsets as bf16x2
        uint32_t sgw[SPI];      // group-wise forward: the stage's scale as bf16x2
        if (ZP && MODE == FUSED_FWD_PC) {
          // per-channel forward: this row's zero offset (dX and the group-wise forward read theirs
          // from the factor slot below)
          const uint32_t z2 = pack_rn_bf16x2(args.zero[row_g], args.zero[row_g]);
#pragma unroll
          for (int j = 0; j < SPI; ++j)
#pragma unroll
            for (int e = 0; e < 8; ++e) zw[j][e] = z2;
        }
        // the stages' stored bases, each read as soon as it has landed
        uint32_t raw[SPI][8];
#pragma unroll
        for (int j = 0; j < SPI; ++j) {
          const uint32_t gj = g + kk + j, fslot = gj % NF;
          ok = wait_bounded(bar(BAR_PFULL + fslot), (gj / NF) & 1u, ctl, 12);
          if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
          const uint32_t fs = smem + OFF_FSLOTS + fslot * FSLOT_BYTES;
          if (PACKED) {
            const uint2 r = ld_shared_v2(fs + swz_offset(row, c >> 1, 32) + 8 * (c & 1));
            raw[j][0] = r.x;
            raw[j][1] = r.y;
          } else if (fmt_16bit(FMT)) {
            const uint4 r0 = ld_shared_v4(fs + swz_offset(row, 2 * c, 128));
            const uint4 r1 = ld_shared_v4(fs + swz_offset(row, 2 * c + 1, 128));
            raw[j][0] = r0.x, raw[j][1] = r0.y, raw[j][2] = r0.z, raw[j][3] = r0.w;
            raw[j][4] = r1.x, raw[j][5] = r1.y, raw[j][6] = r1.z, raw[j][7] = r1.w;
          } else {
            const uint4 r = ld_shared_v4(fs + swz_offset(row, c, 64));
            raw[j][0] = r.x, raw[j][1] = r.y, raw[j][2] = r.z, raw[j][3] = r.w;
          }
          if (MODE == FUSED_DX) {
            // the 16 bf16 scales (zero offsets) of this warp's contraction indices, as bf16x2 words
            const uint4 s0 = ld_shared_v4(fs + PR::FS_X + 32u * c), s1 = ld_shared_v4(fs + PR::FS_X + 32u * c + 16u);
            scw[j][0] = s0.x, scw[j][1] = s0.y, scw[j][2] = s0.z, scw[j][3] = s0.w;
            scw[j][4] = s1.x, scw[j][5] = s1.y, scw[j][6] = s1.z, scw[j][7] = s1.w;
            if (ZP) {
              const uint4 z0 = ld_shared_v4(fs + PR::FS_X + 512u + 32u * c);
              const uint4 z1 = ld_shared_v4(fs + PR::FS_X + 512u + 32u * c + 16u);
              zw[j][0] = z0.x, zw[j][1] = z0.y, zw[j][2] = z0.z, zw[j][3] = z0.w;
              zw[j][4] = z1.x, zw[j][5] = z1.y, zw[j][6] = z1.z, zw[j][7] = z1.w;
            }
          } else if (MODE == FUSED_FWD_GROUP) {
            // this thread's row's scale (and zero offset) in the stage's group, as bf16x2
            const uint32_t sv = ld_shared_u16(fs + PR::FS_X + 2u * row);
            sgw[j] = sv | (sv << 16);
            if (ZP) {
              const uint32_t zv = ld_shared_u16(fs + PR::FS_X + 512u + 2u * row);
#pragma unroll
              for (int e = 0; e < 8; ++e) zw[j][e] = zv | (zv << 16);
            }
          }
        }
        if (!ok) break;
        uint32_t w[SPI][8];
#pragma unroll
        for (int j = 0; j < SPI; ++j) {
          const uint32_t gj = g + kk + j;
          float v[16];
          // the codes base with the clipped codes stored as c + 64: bf16 straight from the bytes
          const bool b64 = NL && args.codes_bias == 64;
          uint32_t c8[8];
          if (b64) {
#pragma unroll
            for (int i = 0; i < 4; ++i) decode_b64_bf16x4(raw[j][i], c8[2 * i], c8[2 * i + 1]);
          } else if (NL && args.codes_bias == 128) {
            decode_ob16(raw[j], v);
          } else {
            decode16<FMT>(raw[j], v);
          }
          float Lv[16];
          if (!NL) {
            const uint32_t lb = gj % NLB;
            ok = wait_bounded(bar(BAR_LFULL + lb), (gj / NLB) & 1u, ctl, 13);
            if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
            tc_fence_after();
            tmem_ld16(tmem + lane_off + COL_L + BK * lb + 16 * c, Lv);
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) report(BAR_LEMPTY + lb, pw);
          }
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            uint32_t cw;
            if (NL) {
              cw = b64                         ? c8[e]
                   : args.codes_bias == 128    ? pack_int_bf16x2(v[2 * e], v[2 * e + 1])
                                               : int_codes_bf16x2(v[2 * e], v[2 * e + 1], qp);
            } else {
              const float2 u = UB ? u_bf16x2(Lv[2 * e], Lv[2 * e + 1], v[2 * e], v[2 * e + 1], lr2)
                                  : __ffma2_rn(make_float2(Lv[2 * e], Lv[2 * e + 1]),
                                               make_float2(qp.lr_scale, qp.lr_scale),
                                               make_float2(v[2 * e], v[2 * e + 1]));
              cw = codes_bf16x2(__fadd2_rn(u, make_float2(qp.magic, qp.magic)), qp);
            }
            if (ZP) cw = sub_bf16x2(cw, zw[j][e]);
            if (MODE == FUSED_FWD_PC) {
              w[j][e] = cw;
            } else {
              w[j][e] = mul_bf16x2(cw, MODE == FUSED_DX ? scw[j][e] : sgw[j]);
            }
          }
        }
        if (!ok) break;
        // Each stage's W_hat buffer (in its token slot) was last read by the product of stage gj - NT.
#pragma unroll
        for (int j = 0; j < SPI; ++j) {
          const uint32_t gj = g + kk + j, ts = gj % NT;
          ok = wait_bounded(bar(BAR_TEMPTY + ts), ((gj / NT) & 1u) ^ 1u, ctl, 14);
          if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
          const uint32_t wt = smem + OFF_TSLOTS + ts * TSLOT_BYTES + TS_W;
          st_shared_v4(wt + swz_offset(row, 2 * c, 128), w[j][0], w[j][1], w[j][2], w[j][3]);
          st_shared_v4(wt + swz_offset(row, 2 * c + 1, 128), w[j][4], w[j][5], w[j][6], w[j][7]);
        }
        if (!ok) break;
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
#pragma unroll
          for (int j = 0; j < SPI; ++j) {
            const uint32_t gj = g + kk + j;
            report(BAR_TFULL + gj % NT, pw);
            mbar_arrive(bar(BAR_FEMPTY + gj % NF));
          }
        }
      }
      if (!ok) break;
      // ------------------------------------------------------------ epilogue
      float scale = 1.0f;
      if (MODE == FUSED_FWD_PC) scale = args.s[row_g];
      if (MODE != FUSED_DX && args.s_x != nullptr) scale *= *args.s_x;
      ok = wait_spin_bounded(bar(BAR_ACCFULL), it & 1u, ctl, 15);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      const bool odd = lane & 1;
#pragma unroll 1
      for (int ch = 0; ch < EPI_COLS / 16; ++ch) {
        float acc[16];
        const int col = c * EPI_COLS + 16 * ch;   // accumulator column = token offset in the tile
        tmem_ld16(tmem + lane_off + col, acc);
        tmem_ld_wait();
        const int tok0 = tb * BTP + col;
        uint32_t mword = 0xffffffffu;
        if (MODE == FUSED_DX && args.xmask != nullptr && tok0 < args.T)
          mword = args.xmask[static_cast<int64_t>(row_g) * args.xmask_ld + tok0 / 32] >> (tok0 & 31);
#pragma unroll
        for (int e = 0; e < 16; ++e) acc[e] = ((mword >> e) & 1u) ? acc[e] * scale : 0.0f;
        store_row_pairs_bf16(acc, odd, args.out, args.out_ld, row_g, tok0, args.T);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) report(BAR_ACCEMPTY, pw);
      g += nk;
      ++it;
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // neither CTA leaves while the other may still read its shared memory
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

template <int MODE, int FMT, bool ZP, bool UB, bool NL>
cudaError_t launch_pair_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                            const FusedArgs& args, int npairs, cudaStream_t stream) {
  constexpr uint32_t smem = PairRing<FMT, NL, MODE == FUSED_DX || MODE == FUSED_FWD_GROUP>::SMEM_BYTES;
  static bool configured[kMaxDevices] = {};
  const void* fn = reinterpret_cast<const void*>(fused_pair_kernel<MODE, FMT, ZP, UB, NL>);
  cudaError_t e = ensure_smem_attr(fn, static_cast<int>(smem), configured);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(2 * npairs), 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // The persistent grid holds no more pairs than can be resident at once (an SM that has no
  // partner in its GPC cannot host half of a pair), looked up once per device.
  static int max_pairs[kMaxDevices] = {};
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (max_pairs[dev] == 0) {
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, fused_pair_kernel<MODE, FMT, ZP, UB, NL>, &cfg);
    if (e != cudaSuccess) return e;
    if (n < 1) return cudaErrorInvalidConfiguration;
    max_pairs[dev] = n;
  }
  if (npairs > max_pairs[dev]) {
    npairs = max_pairs[dev];
    cfg.gridDim = dim3(static_cast<unsigned>(2 * npairs), 1, 1);
  }
  e = cudaLaunchKernelEx(&cfg, fused_pair_kernel<MODE, FMT, ZP, UB, NL>, a, b, c, d, args);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int MODE, int FMT>
cudaError_t launch_pair_fmt(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                            const FusedArgs& args, int npairs, cudaStream_t stream) {
  if (args.r16 == 0) {
    if (FMT != FMT_Q8 || args.u_bf16) return cudaErrorInvalidValue;
    return args.zero != nullptr ? launch_pair_one<MODE, FMT_Q8, true, false, true>(a, b, c, d, args, npairs, stream)
                                : launch_pair_one<MODE, FMT_Q8, false, false, true>(a, b, c, d, args, npairs, stream);
  }
  if (args.u_bf16) {
    if (FMT == FMT_F16 || args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_pair_one<MODE, FMT == FMT_F16 ? FMT_Q8 : FMT, false, true, false>(a, b, c, d, args, npairs, stream);
  }
  if (fmt_float(FMT)) {
    if (args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_pair_one<MODE, FMT, false, false, false>(a, b, c, d, args, npairs, stream);
  }
  return args.zero != nullptr ? launch_pair_one<MODE, FMT, true, false, false>(a, b, c, d, args, npairs, stream)
                              : launch_pair_one<MODE, FMT, false, false, false>(a, b, c, d, args, npairs, stream);
}

template <int MODE>
cudaError_t launch_pair_mode(int fmt, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                             const CUtensorMap& d, const FusedArgs& args, int npairs, cudaStream_t stream) {
  switch (fmt) {
    case FMT_Q8: return launch_pair_fmt<MODE, FMT_Q8>(a, b, c, d, args, npairs, stream);
    case FMT_I4:
      if (MODE == FUSED_DX) return cudaErrorInvalidValue;
      return launch_pair_fmt<MODE, MODE == FUSED_DX ? FMT_Q8 : FMT_I4>(a, b, c, d, args, npairs, stream);
    case FMT_BF16: return launch_pair_fmt<MODE, FMT_BF16>(a, b, c, d, args, npairs, stream);
    case FMT_F16: return launch_pair_fmt<MODE, FMT_F16>(a, b, c, d, args, npairs, stream);
    case FMT_E4M3: return launch_pair_fmt<MODE, FMT_E4M3>(a, b, c, d, args, npairs, stream);
    case FMT_E5M2: return launch_pair_fmt<MODE, FMT_E5M2>(a, b, c, d, args, npairs, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_fused_pair(int mode, int fmt, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi,
                              const CUtensorMap& tm_rf, const CUtensorMap& tm_sf, const FusedArgs& args, int npairs,
                              cudaStream_t stream) {
  if (npairs < 1 || (args.kdim % 128) != 0 || args.kdim < 128 || (args.rows % 256) != 0 || args.sf_mn ||
      args.num_rb != args.rows / 128)
    return cudaErrorInvalidValue;
  switch (mode) {
    case FUSED_FWD_PC: return launch_pair_mode<FUSED_FWD_PC>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, npairs, stream);
    case FUSED_FWD_GROUP:
      return launch_pair_mode<FUSED_FWD_GROUP>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, npairs, stream);
    case FUSED_DX: return launch_pair_mode<FUSED_DX>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, npairs, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lrqat
