// Fused LR-QAT GEMM for the forward (Y = X W_hat^T) and the input gradient
// (dX = dY W_hat), with W_hat rebuilt on chip and never stored (Eq. 8 of the
// paper; the recompute replaces the checkpointing of Sec. 3).
//
// One persistent CTA per SM processes tiles of 128 weight rows x 448 tokens,
// one 64-wide slice of the contraction per pipeline stage:
//   * token ring (2 slots): two loader warps, one per slot, bring with TMA the
//     token operand as 2 boxes of 224 x 64 bf16 (128-byte rows, SW128); each slot
//     also holds the bf16 operand tile W_hat of its stage;
//   * factor ring (4 slots; 2 for 16-bit bases): one loader warp brings the stored
//     base (128 x 64 bytes, SW64, for 8-bit formats; packed: 128 x 32 bytes, SW32;
//     BF16/FP16: 128 x 128 bytes, SW128) and a 64-row slice of the second low-rank
//     factor, only its first r16 columns (rows of 32, 64 or 128 bytes, swizzled to
//     the row width);
//   * the MMA warp computes the low-rank tile L = RF * SF^T (M=128, N=64, K=r
//     rounded to 16) into a TMEM buffer, issued ahead of the main product of the
//     previous stage so that it is ready when that product finishes;
//   * sixteen producer warps (lane quarter q = warp % 4, column chunk c of 16)
//     read L with tcgen05.ld, decode the stored base, form
//     u = phi^{-1}(Phi0) + (alpha/r) L with packed fp32 arithmetic, round half to
//     even, clip, (scale) and write W_hat (SW128, K-major) while the previous
//     stage's product runs;
//   * the MMA warp runs the main product, 8 MMAs of M=128, N=224, K=16, into two
//     fp32 TMEM accumulators; the same sixteen warps drain them in the epilogue.
// Forward: rows = m (weight rows), contraction = k, RF = A (padded), SF = B^T.
// dX:      rows = k, contraction = m over the transposed base Phi0^T,
//          RF = B^T (padded), SF = A (padded); the scale varies along the
//          contraction, so the producer emits bf16(s * c).
// Large 128-byte-row boxes matter: an SM's TMA throughput falls with the number
// of boxes it processes, and loads issued by one warp are handled one at a time,
// hence one loader warp per ring slot of the token operand.
// Ranks above 64 (NL): the base operand already holds the codes round(u) of Eq. 8,
// low-rank term included (written once per call by the tensor-core code pass), so no
// factor is loaded and no low-rank tile is computed; the producers clip, (scale) and
// store W_hat from the base alone.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int BN = 224;
constexpr int NACC = 2;
constexpr int BT = BN * NACC;                    // 448 tokens per tile
constexpr int NT = 2;                            // token ring slots
constexpr int NF_MAX = 4;                        // factor ring slots (power of two; 2 for 16-bit bases)
constexpr int NUM_PROD_WARPS = 16;
constexpr int FIRST_TMA_WARP = 2 + NUM_PROD_WARPS;
constexpr int NUM_TMA_WARPS = NT + 1;            // token loaders + factor loader
constexpr int NUM_THREADS = 32 * (FIRST_TMA_WARP + NUM_TMA_WARPS);
constexpr int EPI_COLS = NACC * BN / 4;          // accumulator columns drained per warp (112)

constexpr uint32_t RF_BYTES = 128 * 128;         // 128 rows x 64 rank columns (bf16)
constexpr uint32_t TOK_HALF = BN * 128;          // 224 tokens x 64 bf16
constexpr uint32_t TOK_BYTES = 2 * TOK_HALF;
constexpr uint32_t W_BYTES = 128 * 128;          // 128 rows x 64 bf16
constexpr uint32_t SF_BYTES = 64 * 128;          // 64 slice rows x up to 64 rank columns (bf16)
constexpr uint32_t TSLOT_BYTES = TOK_BYTES + W_BYTES;
constexpr uint32_t OFF_RF = 0;
constexpr uint32_t OFF_TSLOTS = RF_BYTES;
constexpr uint32_t OFF_FSLOTS = OFF_TSLOTS + NT * TSLOT_BYTES;
constexpr uint32_t TS_W = TOK_BYTES;             // offsets inside a token slot

// Factor ring of a storage format: a 16-bit base tile (128 x 64 x 2 bytes) doubles
// the slot, so that ring has 2 slots.
template <int FMT>
struct FactorRing {
  static constexpr int NF = fmt_16bit(FMT) ? 2 : 4;
  static constexpr uint32_t PHI_BYTES = fmt_16bit(FMT) ? 128 * 128 : 128 * 64;   // packed uses half
  static constexpr uint32_t PHI_TX = FMT == FMT_I4 ? PHI_BYTES / 2 : PHI_BYTES;  // bytes one base tile brings
  static constexpr uint32_t FSLOT_BYTES = PHI_BYTES + SF_BYTES;
  static constexpr uint32_t FS_SF = PHI_BYTES;    // offset of the factor slice inside a slot
  static constexpr uint32_t SMEM_BYTES = OFF_FSLOTS + NF * FSLOT_BYTES + 1024;   // + 1 KB for 1024-B alignment
  static_assert(FSLOT_BYTES % 1024 == 0 && FS_SF % 1024 == 0, "swizzled tiles must start on 1024-byte boundaries");
  static_assert(SMEM_BYTES + 512 <= 232448, "shared memory budget");
  static_assert((NF & (NF - 1)) == 0 && NF <= NF_MAX, "factor ring index uses a mask");
};

static_assert(TSLOT_BYTES % 1024 == 0 && TOK_HALF % 1024 == 0 && TS_W % 1024 == 0 && OFF_TSLOTS % 1024 == 0 &&
                  OFF_FSLOTS % 1024 == 0,
              "swizzled tiles must start on 1024-byte boundaries");
static_assert(EPI_COLS % 16 == 0, "epilogue drains 16-column chunks");

constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_L = NACC * BN;            // one 64-column low-rank buffer at 448
static_assert(COL_L + BK <= TMEM_COLS, "TMEM budget");

// barrier indices
constexpr int BAR_TFULL = 0;
constexpr int BAR_TEMPTY = BAR_TFULL + NT;       // main product of the slot finished
constexpr int BAR_WFULL = BAR_TEMPTY + NT;       // W_hat tile of the slot written
constexpr int BAR_FFULL = BAR_WFULL + NT;
constexpr int BAR_FEMPTY = BAR_FFULL + NF_MAX;
constexpr int BAR_LFULL = BAR_FEMPTY + NF_MAX;
constexpr int BAR_LEMPTY = BAR_LFULL + 1;
constexpr int BAR_RFFULL = BAR_LEMPTY + 1;
constexpr int BAR_RFEMPTY = BAR_RFFULL + 1;
constexpr int BAR_ACCFULL = BAR_RFEMPTY + 1;
constexpr int BAR_ACCEMPTY = BAR_ACCFULL + 1;
constexpr int BAR_DRAIN = BAR_ACCEMPTY + 1;
constexpr int NUM_BARS = BAR_DRAIN + 1;

// Bounded wait that ignores the abort flag: used only to let in-flight
// asynchronous copies or MMAs land before the CTA releases its resources.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) break;
  }
}

// Stages are numbered globally over the CTA's tiles (gg); the contraction has an
// even number of slices, so stage gg uses token slot gg % 2 for the (gg / 2)-th
// time and factor slot gg % NF for the (gg / NF)-th time.
// UB: pre-round value in bf16 (u_bf16x2) instead of one fp32 FMA.
// NL: no low-rank term (the base holds the unclipped codes, FMT_Q8 with 0 fraction bits).
template <int MODE, int FMT, bool ZP, bool UB, bool NL>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    fused_gemm_kernel(const __grid_constant__ CUtensorMap tm_tok, const __grid_constant__ CUtensorMap tm_phi,
                      const __grid_constant__ CUtensorMap tm_rf, const __grid_constant__ CUtensorMap tm_sf,
                      const FusedArgs args) {
  using FR = FactorRing<FMT>;
  // forward: the second factor's slice may come MN-major straight from B (compiled out of dX)
  const bool sf_mn = MODE != FUSED_DX && args.sf_mn;
  constexpr int NF = FR::NF;
  constexpr bool PACKED = FMT == FMT_I4;
  constexpr uint32_t FSLOT_BYTES = FR::FSLOT_BYTES;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[NUM_BARS];
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int abort_s;

  const uint32_t smem = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };

  if (threadIdx.x == 0) {
    abort_s = 0;
    for (int s = 0; s < NT; ++s) {
      mbar_init(bar(BAR_TFULL + s), 1);
      mbar_init(bar(BAR_TEMPTY + s), 1);
      mbar_init(bar(BAR_WFULL + s), NUM_PROD_WARPS);
    }
    for (int s = 0; s < NF; ++s) {
      mbar_init(bar(BAR_FFULL + s), 1);
      // Freed by the producers once they have built W_hat of the stage: by then the
      // low-rank MMA that read the factor slice has completed (they waited for it).
      mbar_init(bar(BAR_FEMPTY + s), NUM_PROD_WARPS);
    }
    mbar_init(bar(BAR_LFULL), 1);
    mbar_init(bar(BAR_LEMPTY), NUM_PROD_WARPS);
    mbar_init(bar(BAR_RFFULL), 1);
    mbar_init(bar(BAR_RFEMPTY), 1);
    mbar_init(bar(BAR_ACCFULL), 1);
    mbar_init(bar(BAR_ACCEMPTY), NUM_PROD_WARPS);
    mbar_init(bar(BAR_DRAIN), 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};
  const int nk = args.kdim / BK;   // even, at least 2 (kdim is a multiple of 128)

  if (warp == 0) {
    // ------------------------------------------------- row factor (per tile)
    if (!NL && lane == 0) {
      prefetch_tensormap(&tm_rf);
      uint32_t it = 0;
      for (int tile = blockIdx.x; tile < args.num_tiles; tile += gridDim.x) {
        const int rb = tile % args.num_rb;
        if (!wait_spin_bounded(bar(BAR_RFEMPTY), (it & 1u) ^ 1u, ctl, 1)) break;
        mbar_arrive_expect_tx(bar(BAR_RFFULL), RF_BYTES);
        tma_load_2d(smem + OFF_RF, &tm_rf, 0, rb * BM, bar(BAR_RFFULL));
        ++it;
      }
      if (it > 0) drain_wait(bar(BAR_RFFULL), (it - 1) & 1u, args.timeout_ns);
    }
  } else if (warp >= FIRST_TMA_WARP && warp < FIRST_TMA_WARP + NT) {
    // ------------------------------------------- token loaders (one per slot)
    const uint32_t t = warp - FIRST_TMA_WARP;
    if (lane == 0) prefetch_tensormap(&tm_tok);
    const uint32_t st = smem + OFF_TSLOTS + t * TSLOT_BYTES;
    const uint32_t fb = bar(BAR_TFULL + t), eb = bar(BAR_TEMPTY + t);
    uint32_t n = 0;   // uses of this slot so far
    bool ok = true;
    for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
      const int tb = tile / args.num_rb;
      for (int kk = t; kk < nk; kk += NT) {
        if (lane == 0) ok = wait_spin_bounded(eb, (n & 1u) ^ 1u, ctl, 2);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0) mbar_arrive_expect_tx(fb, TOK_BYTES);
        __syncwarp();
        if (lane == 0) tma_load_2d(st, &tm_tok, kk * BK, tb * BT, fb);
        if (lane == 1) tma_load_2d(st + TOK_HALF, &tm_tok, kk * BK, tb * BT + BN, fb);
        ++n;
      }
    }
    // Let every issued copy land before the CTA can exit.
    if (lane == 0 && n > 0) drain_wait(fb, (n - 1) & 1u, args.timeout_ns);
  } else if (warp == FIRST_TMA_WARP + NT) {
    // ------------------------------------------------- factor-ring loader
    if (lane == 0) {
      prefetch_tensormap(&tm_phi);
      prefetch_tensormap(&tm_sf);
    }
    const uint32_t tx = FR::PHI_TX + (NL ? 0u : static_cast<uint32_t>(BK * 2 * (sf_mn ? args.r16 : args.sf_cols)));
    uint32_t gg = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
      const int rb = tile % args.num_rb;
      for (int kk = 0; kk < nk; ++kk, ++gg) {
        const uint32_t s = gg & (NF - 1);
        const uint32_t fb = bar(BAR_FFULL + s);
        if (lane == 0) ok = wait_spin_bounded(bar(BAR_FEMPTY + s), ((gg / NF) & 1u) ^ 1u, ctl, 3);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0) mbar_arrive_expect_tx(fb, tx);
        __syncwarp();
        const uint32_t fs = smem + OFF_FSLOTS + s * FSLOT_BYTES;
        if (lane == 0) tma_load_2d(fs, &tm_phi, PACKED ? kk * (BK / 2) : kk * BK, rb * BM, fb);
        if (!NL && lane == 1) {
          if (sf_mn) tma_load_2d(fs + FR::FS_SF, &tm_sf, kk * BK, 0, fb);   // B rows, 64 columns
          else tma_load_2d(fs + FR::FS_SF, &tm_sf, 0, kk * BK, fb);
        }
      }
    }
    if (lane == 0 && gg > 0) {
      const uint32_t last = gg - 1;
      drain_wait(bar(BAR_FFULL + (last & (NF - 1))), (last / NF) & 1u, args.timeout_ns);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      // This thread's instruction stream sits between consecutive MMAs, so keep it
      // short: descriptors of slot 0 are built once; a slot adds its byte stride / 16
      // to the encoded start address and a 16-element K step adds 32 bytes (2 units).
      const uint32_t idesc_main = make_idesc_bf16(128, BN, 0, 0);
      const uint32_t idesc_l = make_idesc_bf16(128, BK, 0, sf_mn ? 1 : 0);
      const int lsteps = args.r16 / 16;
      constexpr uint32_t TSLOT_D = TSLOT_BYTES >> 4, FSLOT_D = FSLOT_BYTES >> 4, TOKH_D = TOK_HALF >> 4;
      // K-major operands advance 32 bytes (2 units) per 16-element K step; MN-major ones
      // (SW128, 8-row atoms of 128-byte rows) advance 16 rows, 2048 bytes (128 units).
      const uint64_t d_rf = make_sdesc(smem + OFF_RF, 16, 1024, SWZ_128B);
      // The K-major factor slice has rows of sf_cols bf16 (32, 64 or 128 bytes, swizzled to
      // match); the MN-major one rows of 64 bf16.
      const uint32_t sf_swz = sf_mn || args.sf_cols == 64 ? SWZ_128B : args.sf_cols == 32 ? SWZ_64B : SWZ_32B;
      const uint64_t d_sf0 = sf_mn ? make_sdesc(smem + OFF_FSLOTS + FR::FS_SF, 128u * args.r16, 1024, sf_swz)
                                   : make_sdesc(smem + OFF_FSLOTS + FR::FS_SF, 16, 16u * args.sf_cols, sf_swz);
      const uint32_t sf_step = sf_mn ? 128u : 2u;
      const uint64_t sk1 = sf_step, sk2 = 2 * sf_step, sk3 = 3 * sf_step;
      const uint64_t d_w0 = make_sdesc(smem + OFF_TSLOTS + TS_W, 16, 1024, SWZ_128B);
      const uint64_t d_tok0 = make_sdesc(smem + OFF_TSLOTS, 16, 1024, SWZ_128B);
      uint32_t g = 0;
      uint32_t it = 0;
      bool ok = true;
      // Low-rank tile of stage gg into the TMEM buffer, once its factor slice has
      // landed and the producers have read the tile of stage gg - 1.
      auto issue_lowrank = [&](uint32_t gg) -> bool {
        const uint32_t s = gg & (NF - 1);
        if (!wait_spin_bounded(bar(BAR_FFULL + s), (gg / NF) & 1u, ctl, 4)) return false;
        if (!wait_spin_bounded(bar(BAR_LEMPTY), (gg & 1u) ^ 1u, ctl, 5)) return false;
        tc_fence_after();
        const uint64_t sf = d_sf0 + s * FSLOT_D;
        const uint32_t dl = tmem + COL_L;
        mma_bf16(dl, d_rf, sf, idesc_l, 0u);
        if (lsteps > 1) mma_bf16(dl, d_rf + 2, sf + sk1, idesc_l, 1u);
        if (lsteps > 2) mma_bf16(dl, d_rf + 4, sf + sk2, idesc_l, 1u);
        if (lsteps > 3) mma_bf16(dl, d_rf + 6, sf + sk3, idesc_l, 1u);
        mma_commit(bar(BAR_LFULL));
        return true;
      };
      for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
        if (!NL && !(ok = wait_spin_bounded(bar(BAR_RFFULL), it & 1u, ctl, 6))) break;
        if (!NL && !(ok = issue_lowrank(g))) break;
        if (!(ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 7))) break;
        tc_fence_after();
        for (int kk = 0; kk < nk; ++kk) {
          const uint32_t gg = g + kk;
          const uint32_t s = gg & 1u, ph = (gg >> 1) & 1u;
          // The low-rank tile of the next stage goes into the tensor pipe ahead of this
          // stage's product as soon as the producers have read the current one, so the
          // W_hat build of the next stage overlaps this product.
          if (!NL && kk + 1 < nk) {
            if (!(ok = issue_lowrank(gg + 1))) break;
            if (kk + 2 == nk) mma_commit(bar(BAR_RFEMPTY));   // last read of the row factor issued
          }
          if (!(ok = wait_spin_bounded(bar(BAR_WFULL + s), ph, ctl, 8))) break;
          if (!(ok = wait_spin_bounded(bar(BAR_TFULL + s), ph, ctl, 9))) break;
          tc_fence_after();
          const uint64_t w = d_w0 + s * TSLOT_D, t = d_tok0 + s * TSLOT_D;
          const uint32_t acc = kk > 0 ? 1u : 0u;
          static_assert(NACC == 2 && BK == 64, "issue sequence below is written for 2 accumulators x 4 K steps");
          mma_bf16(tmem, w, t, idesc_main, acc);
          mma_bf16(tmem, w + 2, t + 2, idesc_main, 1u);
          mma_bf16(tmem, w + 4, t + 4, idesc_main, 1u);
          mma_bf16(tmem, w + 6, t + 6, idesc_main, 1u);
          mma_bf16(tmem + BN, w, t + TOKH_D, idesc_main, acc);
          mma_bf16(tmem + BN, w + 2, t + TOKH_D + 2, idesc_main, 1u);
          mma_bf16(tmem + BN, w + 4, t + TOKH_D + 4, idesc_main, 1u);
          mma_bf16(tmem + BN, w + 6, t + TOKH_D + 6, idesc_main, 1u);
          mma_commit(bar(BAR_TEMPTY + s));
        }
        if (!ok) break;
        mma_commit(bar(BAR_ACCFULL));
        g += nk;
        ++it;
      }
      mma_commit(bar(BAR_DRAIN));
      drain_wait(bar(BAR_DRAIN), 0, args.timeout_ns);
    }
  } else {
    // ------------------------------------------- W_hat producers + epilogue
    const int pw = warp - 2;              // 0..15
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int c = pw >> 2;                // 16-column chunk of the 64-wide slice (and epilogue block)
    const int row = q * 32 + lane;        // row of the tile handled by this thread
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const QuantParams qp = args.q;
    const uint32_t lr2 = pack_rn_bf16x2(qp.lr_scale, qp.lr_scale);   // exact: a power of two when UB
    constexpr bool zp = ZP;   // zero offsets (asymmetric weights): args.zero != nullptr
    uint32_t g = 0;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
      const int rb = tile % args.num_rb;
      const int tb = tile / args.num_rb;
      const int row_g = rb * BM + row;
      for (int kk = 0; kk < nk; ++kk) {
        const uint32_t gg = g + kk;
        // Scales that multiply the operand (group-wise forward, dX), and the zero offsets
        // subtracted from the codes (asymmetric weights) as bf16 pairs.
        float sc[16];
        uint32_t scw[8];   // dX: bf16x2 scales
        uint32_t zw[8];
        if (zp) {
          if (MODE == FUSED_DX) {
            // 16 consecutive bf16 zero offsets of this stage's contraction indices
            const uint16_t* zp = args.z_bf16 + (args.s_ld ? static_cast<int64_t>(row_g / args.group_size) * args.kdim : 0) +
                                 kk * BK + 16 * c;
            const uint4 z0 = __ldg(reinterpret_cast<const uint4*>(zp));
            const uint4 z1 = __ldg(reinterpret_cast<const uint4*>(zp) + 1);
            zw[0] = z0.x, zw[1] = z0.y, zw[2] = z0.z, zw[3] = z0.w;
            zw[4] = z1.x, zw[5] = z1.y, zw[6] = z1.z, zw[7] = z1.w;
          } else {
            const float zr = MODE == FUSED_FWD_GROUP
                                 ? args.zero[static_cast<int64_t>(row_g) * args.s_ld + (kk * BK) / args.group_size]
                                 : args.zero[row_g];
            const uint32_t z2 = pack_rn_bf16x2(zr, zr);
#pragma unroll
            for (int e = 0; e < 8; ++e) zw[e] = z2;
          }
        }
        if (MODE == FUSED_FWD_GROUP) {
          const float v = args.s[static_cast<int64_t>(row_g) * args.s_ld + (kk * BK) / args.group_size];
#pragma unroll
          for (int e = 0; e < 16; ++e) sc[e] = v;
        } else if (MODE == FUSED_DX) {
          // 16 consecutive bf16 scales of this stage's contraction indices, as bf16x2 words
          const uint16_t* sp = args.s_bf16 + (args.s_ld ? static_cast<int64_t>(row_g / args.group_size) * args.kdim : 0) +
                               kk * BK + 16 * c;
          const uint4 s0 = __ldg(reinterpret_cast<const uint4*>(sp));
          const uint4 s1 = __ldg(reinterpret_cast<const uint4*>(sp) + 1);
          scw[0] = s0.x, scw[1] = s0.y, scw[2] = s0.z, scw[3] = s0.w;
          scw[4] = s1.x, scw[5] = s1.y, scw[6] = s1.z, scw[7] = s1.w;
        }
        // The stored base usually lands well before the low-rank tile: decode it first,
        // keeping the low-rank read -> W_hat chain short.
        const uint32_t fslot = gg & (NF - 1);
        ok = wait_bounded(bar(BAR_FFULL + fslot), (gg / NF) & 1u, ctl, 11);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        const uint32_t fs = smem + OFF_FSLOTS + fslot * FSLOT_BYTES;
        float v[16];
        uint32_t raw[8];
        if (PACKED) {
          const uint2 r = ld_shared_v2(fs + swz_offset(row, c >> 1, 32) + 8 * (c & 1));
          raw[0] = r.x;
          raw[1] = r.y;
        } else if (fmt_16bit(FMT)) {
          // 16 values = 32 bytes of a 128-byte row: 16-byte chunks 2c and 2c + 1 (SW128)
          const uint4 r0 = ld_shared_v4(fs + swz_offset(row, 2 * c, 128));
          const uint4 r1 = ld_shared_v4(fs + swz_offset(row, 2 * c + 1, 128));
          raw[0] = r0.x, raw[1] = r0.y, raw[2] = r0.z, raw[3] = r0.w;
          raw[4] = r1.x, raw[5] = r1.y, raw[6] = r1.z, raw[7] = r1.w;
        } else {
          const uint4 r = ld_shared_v4(fs + swz_offset(row, c, 64));
          raw[0] = r.x, raw[1] = r.y, raw[2] = r.z, raw[3] = r.w;
        }
        // the codes base with the clipped codes stored as c + 64: bf16 straight from the bytes
        const bool b64 = NL && args.codes_bias == 64;
        uint32_t c8[8];
        if (b64) {
#pragma unroll
          for (int i = 0; i < 4; ++i) decode_b64_bf16x4(raw[i], c8[2 * i], c8[2 * i + 1]);
        } else if (NL && args.codes_bias == 128) {
          decode_ob16(raw, v);
        } else {
          decode16<FMT>(raw, v);
        }
        float Lv[16];
        if (!NL) {
          ok = wait_bounded(bar(BAR_LFULL), gg & 1u, ctl, 10);
          if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
          tc_fence_after();
          tmem_ld16(tmem + lane_off + COL_L + 16 * c, Lv);
          tmem_ld_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(BAR_LEMPTY));
        }
        uint32_t w[8];
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
                                             make_float2(qp.lr_scale, qp.lr_scale), make_float2(v[2 * e], v[2 * e + 1]));
            cw = codes_bf16x2(__fadd2_rn(u, make_float2(qp.magic, qp.magic)), qp);
          }
          if (zp) cw = sub_bf16x2(cw, zw[e]);   // c - z, exact small integers
          if (MODE == FUSED_FWD_PC) {
            w[e] = cw;
          } else {
            // bf16(bf16(s) * c): the exact bf16 codes times the bf16-rounded scales,
            // one packed multiply instead of an fp32 clip, multiply and conversion.
            w[e] = mul_bf16x2(cw, MODE == FUSED_DX ? scw[e] : pack_rn_bf16x2(sc[2 * e], sc[2 * e + 1]));
          }
        }
        // The W_hat buffer of this token slot was last read by the product of stage gg - 2.
        const uint32_t ts = gg & 1u;
        ok = wait_bounded(bar(BAR_TEMPTY + ts), ((gg >> 1) & 1u) ^ 1u, ctl, 12);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        const uint32_t wt = smem + OFF_TSLOTS + ts * TSLOT_BYTES + TS_W;
        st_shared_v4(wt + swz_offset(row, 2 * c, 128), w[0], w[1], w[2], w[3]);
        st_shared_v4(wt + swz_offset(row, 2 * c + 1, 128), w[4], w[5], w[6], w[7]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(bar(BAR_WFULL + ts));
          mbar_arrive(bar(BAR_FEMPTY + fslot));
        }
      }
      if (!ok) break;
      // ------------------------------------------------------------ epilogue
      float scale = 1.0f;
      if (MODE == FUSED_FWD_PC) scale = args.s[row_g];
      if (MODE != FUSED_DX && args.s_x != nullptr) scale *= *args.s_x;
      // polled: the drain, and with it the next tile's start, follows this phase directly
      ok = wait_spin_bounded(bar(BAR_ACCFULL), it & 1u, ctl, 13);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      const bool odd = lane & 1;
#pragma unroll 1
      for (int ch = 0; ch < EPI_COLS / 16; ++ch) {
        float acc[16];
        const int col = c * EPI_COLS + 16 * ch;   // accumulator column = token offset in the tile
        tmem_ld16(tmem + lane_off + col, acc);
        tmem_ld_wait();
        const int tok0 = tb * BT + col;
        uint32_t mword = 0xffffffffu;
        if (MODE == FUSED_DX && args.xmask != nullptr && tok0 < args.T)
          mword = args.xmask[static_cast<int64_t>(row_g) * args.xmask_ld + tok0 / 32] >> (tok0 & 31);
#pragma unroll
        for (int e = 0; e < 16; ++e) acc[e] = ((mword >> e) & 1u) ? acc[e] * scale : 0.0f;
        store_row_pairs_bf16(acc, odd, args.out, args.out_ld, row_g, tok0, args.T);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(BAR_ACCEMPTY));
      g += nk;
      ++it;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int MODE, int FMT, bool ZP, bool UB, bool NL = false>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                       const FusedArgs& args, int grid, cudaStream_t stream) {
  constexpr uint32_t smem = FactorRing<FMT>::SMEM_BYTES;
  static bool configured[kMaxDevices] = {};
  const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(fused_gemm_kernel<MODE, FMT, ZP, UB, NL>),
                                         static_cast<int>(smem), configured);
  if (e != cudaSuccess) return e;
  fused_gemm_kernel<MODE, FMT, ZP, UB, NL><<<grid, NUM_THREADS, smem, stream>>>(a, b, c, d, args);
  return cudaGetLastError();
}

// The operand of the dX product is the transposed base, never packed (the transpose
// unpacks nibbles into bytes).  Zero offsets exist only with the integer formats; the
// bf16 pre-round value only without them and with bases exact in bf16 (not FP16).
template <int MODE, int FMT>
cudaError_t launch_fmt(const CUtensorMap& tm_tok, const CUtensorMap& tm_phi, const CUtensorMap& tm_rf,
                       const CUtensorMap& tm_sf, const FusedArgs& args, int grid, cudaStream_t stream) {
  if (args.u_bf16) {
    if (FMT == FMT_F16 || args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_one<MODE, FMT == FMT_F16 ? FMT_Q8 : FMT, false, true>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid,
                                                                          stream);
  }
  if (fmt_float(FMT)) {
    if (args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_one<MODE, FMT, false, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
  }
  return args.zero != nullptr ? launch_one<MODE, FMT, true, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream)
                              : launch_one<MODE, FMT, false, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
}

template <int MODE>
cudaError_t launch_mode(int fmt, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi, const CUtensorMap& tm_rf,
                        const CUtensorMap& tm_sf, const FusedArgs& args, int grid, cudaStream_t stream) {
  if (args.r16 == 0) {
    // no low-rank term: the base holds int8 codes (0 fraction bits), the bf16 pre-round value
    // (if any) was applied when they were written
    if (fmt != FMT_Q8 || args.u_bf16) return cudaErrorInvalidValue;
    return args.zero != nullptr ? launch_one<MODE, FMT_Q8, true, false, true>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream)
                                : launch_one<MODE, FMT_Q8, false, false, true>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
  }
  switch (fmt) {
    case FMT_Q8: return launch_fmt<MODE, FMT_Q8>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FMT_I4:
      if (MODE == FUSED_DX) return cudaErrorInvalidValue;
      return launch_fmt<MODE, MODE == FUSED_DX ? FMT_Q8 : FMT_I4>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FMT_BF16: return launch_fmt<MODE, FMT_BF16>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FMT_F16: return launch_fmt<MODE, FMT_F16>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FMT_E4M3: return launch_fmt<MODE, FMT_E4M3>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FMT_E5M2: return launch_fmt<MODE, FMT_E5M2>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int fused_smem_bytes(int fmt) {
  return static_cast<int>(fmt_16bit(fmt) ? FactorRing<FMT_BF16>::SMEM_BYTES : FactorRing<FMT_Q8>::SMEM_BYTES);
}

cudaError_t launch_fused(int mode, int fmt, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi,
                         const CUtensorMap& tm_rf, const CUtensorMap& tm_sf, const FusedArgs& args, int grid,
                         cudaStream_t stream) {
  if (grid < 1 || (args.kdim % 128) != 0 || args.kdim < 128) return cudaErrorInvalidValue;
  switch (mode) {
    case FUSED_FWD_PC: return launch_mode<FUSED_FWD_PC>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FUSED_FWD_GROUP:
      return launch_mode<FUSED_FWD_GROUP>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FUSED_DX: return launch_mode<FUSED_DX>(fmt, tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lrqat
