// Fused weight-gradient kernel on CTA pairs (ranks up to 64).  The same computation as the
// one-SM kernel (dw.cu): for a tile of weight rows i x 256 columns j and a range of tokens
//   G = dY^T X_hat                 (tcgen05, fp32 accumulator in TMEM, never stored)
// and, in the epilogue, the straight-through gradients of Eq. 8:
//   u = phi^{-1}(Phi0) + (alpha/r) A B,  M = 1[n <= round(u) <= p],  c = clip(round(u), n, p)
//   dU = G * s * M,  dA_partial = dU B^T,  dB^T_partial = dU^T A,  ds_partial = sum_j G * c.
//
// Why this shape: each SM of a pair loads its own 128 rows of dY and half of the 256 X columns
// per stage (the one-SM kernel's 128 x 256 tile loads all 256 columns), and a stage holds 64
// tokens, four K steps between two barrier handshakes instead of two.  Measured on a
// 4096 x 4096 layer at T = 8192: one-SM kernel 229 us, pairs with 32-token stages 225 us, pairs
// with 64-token stages 201 us (three stages of 64 tokens: 242 us; four are kept in flight).
//
// Tile of a pair: rows 256 ib .. (CTA rank c: 128 c .. 128 c + 127 of them), columns 256 jt ..,
// processed in two chunks of 128 columns.  Every MMA of the kernel is a pair MMA (a kernel may
// not mix one-SM and pair MMAs):
//   G:    M = 256 rows i, N = 256 columns j (each CTA holds 128 of the X columns), K = tokens
//         (4 K steps of 16 per 64-token stage);
//   L:    M = 256 rows i, N = 128 columns of the chunk (64 per CTA), K = r16;
//   dA:   M = 256 rows i, N = r16 (each CTA holds half of the ranks of the chunk's B slice),
//         K = 128 columns j of the chunk;
//   dB^T: each CTA's own partial over its 128 rows: M = 256 with rows = the chunk's columns j
//         of each CTA's dU^T, N = r16 (half of the ranks per CTA), K = the 128 rows of one
//         CTA; issued twice, against A's rows of CTA 0 with CTA 1's output lanes disabled and
//         against those of CTA 1 with CTA 0's disabled, so that each CTA's TMEM receives the
//         partial over its own rows, written out like the one-SM kernel's.
// The partial outputs are laid out as the one-SM kernel's (per 128-row block), so the same
// reduction sums them.
//
// Roles (480 threads per CTA): warp 0 loads the epilogue operands, warp 1 owns TMEM and (in
// the leader, rank 0) issues the main loop's MMAs, warps 2..9 run the epilogue, warps 10..13
// fill the stages (one box of every stage each), warp 14 (in the leader) issues the epilogue's
// MMAs (low-rank tiles and adapter contractions).  Loads that the MMAs read complete on the leader's barriers (both CTAs' bytes);
// the leader waits for the peer's "dU written" and "accumulator drained" events, which each
// peer warp reports with a 16-byte copy into the leader's shared memory.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int NS = 4;
constexpr int BKT = 64;                        // tokens per pipeline stage
constexpr int NUM_EPI_WARPS = 8;
constexpr int NUM_LOADERS = 4;                 // one per box of a stage
constexpr int FIRST_LOADER = 2 + NUM_EPI_WARPS;
constexpr int EPI_MMA_WARP = FIRST_LOADER + NUM_LOADERS;   // the leader's epilogue MMAs
constexpr int NUM_THREADS = 32 * (EPI_MMA_WARP + 1);
constexpr uint32_t SIG_TX = 16u * NUM_EPI_WARPS;   // bytes of the peer's per-warp signals

constexpr uint32_t BOX_BYTES = 64 * BKT * 2;   // one 64-column x 64-token bf16 box (SW128)
constexpr uint32_t STAGE_DY = 2 * BOX_BYTES;   // this CTA's 128 rows i
constexpr uint32_t STAGE_BYTES = STAGE_DY + 2 * BOX_BYTES;   // + its 128 of the 256 columns j
constexpr uint32_t OFF_STAGES = 0;
// A^T [r16 rank rows, this CTA's 128 rows i] (2 boxes of 64 i): MN-major A operand of L.
constexpr uint32_t OFF_AT = OFF_STAGES + NS * STAGE_BYTES;
// A^T [this CTA's r16 / 2 ranks, rows i of CTA 0 | of CTA 1] (2 x 2 boxes of 64 i): the K-major
// B operands of the two dB^T products.
constexpr uint32_t OFF_ATH = OFF_AT + 16384;
constexpr uint32_t OFF_PHI = OFF_ATH + 16384;  // Phi0 chunk 128 x 128 (packed: 128 x 64 B)
// B (padded) [r16 rank rows, this CTA's 64 columns of the chunk]: MN-major B operand of L.
constexpr uint32_t OFF_BPL = OFF_PHI + 16384;
// B (padded) [this CTA's r16 / 2 ranks, the chunk's 128 columns] (2 boxes): K-major B of dA.
constexpr uint32_t OFF_BPA = OFF_BPL + 8192;
constexpr uint32_t OFF_DU = OFF_BPA + 8192;    // dU chunk: 2 atom columns of 128 rows x 128 B
constexpr uint32_t SMEM_TILES = OFF_DU + 32768;
constexpr uint32_t SMEM_BYTES = SMEM_TILES + 1024;
static_assert(SMEM_BYTES + 1024 <= 232448, "shared memory budget");
static_assert(OFF_AT % 1024 == 0 && OFF_BPL % 1024 == 0 && OFF_BPA % 1024 == 0 && OFF_DU % 1024 == 0,
              "swizzled tiles start on 1024-byte boundaries");

constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_G = 0;      // 256 columns
constexpr uint32_t COL_L = 256;    // 128 columns
constexpr uint32_t COL_DA = 384;   // up to 64 columns
constexpr uint32_t COL_DBT = 448;  // up to 64 columns

constexpr int BAR_FULL = 0;                    // leader: both CTAs' stage landed
constexpr int BAR_EMPTY = BAR_FULL + NS;       // both: the stage's MMAs finished
constexpr int BAR_EFFULL = BAR_EMPTY + NS;     // leader: both CTAs' A^T slices of the unit landed
constexpr int BAR_EFEMPTY = BAR_EFFULL + 1;    // both: the unit's MMAs that read them finished
constexpr int BAR_ECFULL = BAR_EFEMPTY + 1;    // leader: both CTAs' B slices of the chunk landed
constexpr int BAR_ECEMPTY = BAR_ECFULL + 1;    // both: the chunk's MMAs finished (base chunk read)
constexpr int BAR_PFULL = BAR_ECEMPTY + 1;     // both: this CTA's base chunk landed
constexpr int BAR_ACCFULL = BAR_PFULL + 1;     // both: G complete
constexpr int BAR_ACCEMPTY = BAR_ACCFULL + 1;  // leader: both CTAs read G
constexpr int BAR_LFULL = BAR_ACCEMPTY + 1;    // both: L of the chunk complete
constexpr int BAR_DUFULL = BAR_LFULL + 1;      // leader: both CTAs wrote dU of the chunk
constexpr int BAR_DBFULL = BAR_DUFULL + 1;     // both: dA / dB^T of the chunk complete
constexpr int BAR_DRAIN = BAR_DBFULL + 1;        // the main-loop MMAs' last completion
constexpr int BAR_DRAIN_E = BAR_DRAIN + 1;       // the epilogue MMAs' last completion
constexpr int NUM_BARS = BAR_DRAIN_E + 1;

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) break;
  }
}

// Pair MMA whose output lanes of one CTA are left untouched: `cta` = 0 writes only CTA 0's
// 128 lanes, 1 only CTA 1's (the mask's words 0-3 cover the lanes of CTA 0, 4-7 those of CTA 1).
__device__ __forceinline__ void mma_bf16_pair_half(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                   uint32_t accumulate, int cta) {
  const uint32_t m0 = cta == 0 ? 0u : 0xffffffffu, m1 = cta == 0 ? 0xffffffffu : 0u;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, {%5, %5, %5, %5, %6, %6, %6, %6}, p;\n\t}"
      ::"r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate), "r"(m0), "r"(m1)
      : "memory");
}

struct Unit {
  int ib, jt, sp, t0, nsteps;   // ib: 256-row block of the pair
  int rev;                      // stages in descending token order
};

__device__ __forceinline__ Unit decode_unit(int u, const DwArgs& a) {
  Unit x;
  x.ib = u % a.ni;
  x.jt = (u / a.ni) % a.nj;
  x.sp = u / (a.ni * a.nj);
  x.t0 = x.sp * a.tchunk;
  int t1 = x.t0 + a.tchunk;
  if (t1 > a.T) t1 = a.T;
  x.nsteps = (t1 - x.t0 + BKT - 1) / BKT;
  x.rev = 0;
  return x;
}

// Whole pair tile number u in processing order: groups of kColGroup column tiles with the
// column tile varying fastest (as in dw.cu).
constexpr int64_t kColGroup = 8;
__device__ __forceinline__ void dw_whole_tile(int64_t u, int ni, int64_t full_tiles, int& ib, int& jt) {
  const int64_t grouped = full_tiles / ni / kColGroup * kColGroup * ni;
  if (u < grouped) {
    const int64_t grp = u / (kColGroup * ni), r = u % (kColGroup * ni);
    jt = static_cast<int>(grp * kColGroup + r % kColGroup);
    ib = static_cast<int>(r / kColGroup);
  } else {
    ib = static_cast<int>(u % ni);
    jt = static_cast<int>(u / ni);
  }
}

// This pair's units (equal token splits, round robin over the pairs), or (tail schedule) its
// whole tiles of the full waves followed by its one part of a tail tile.
struct WorkIter {
  int64_t u;
  bool tail;
};

__device__ __forceinline__ WorkIter work_begin(const DwArgs& a, int pair) {
  return {static_cast<int64_t>(pair), a.sched.tail != 0 && pair < a.sched.tail_grid};
}

__device__ __forceinline__ bool work_next(WorkIter& it, const DwArgs& a, int pair, int npairs, Unit& x) {
  // Odd waves run their stages in descending token order: a wave shares its column (or row) blocks
  // with the wave before it, whose last stages are then still in L2 when it starts.
  if (!a.sched.tail) {
    if (it.u >= a.num_units) return false;
    x = decode_unit(static_cast<int>(it.u), a);
    x.rev = static_cast<int>((it.u / npairs) & 1);
    it.u += npairs;
    return true;
  }
  if (it.u < a.sched.full_tiles) {
    dw_whole_tile(it.u, a.ni, a.sched.full_tiles, x.ib, x.jt);
    x.sp = 0;
    x.t0 = 0;
    x.nsteps = static_cast<int>(a.sched.tsteps);
    x.rev = static_cast<int>((it.u / npairs) & 1);
    it.u += npairs;
    return true;
  }
  if (!it.tail) return false;
  it.tail = false;
  int64_t t;
  int j, q;
  dw_tail_part(pair, a.sched, t, j, q);
  const int64_t tile = a.sched.full_tiles + t;
  const int64_t s0 = j * a.sched.tsteps / q, s1 = (j + 1) * a.sched.tsteps / q;
  x.ib = static_cast<int>(tile % a.ni);
  x.jt = static_cast<int>(tile / a.ni);
  x.sp = j;
  x.t0 = static_cast<int>(s0 * BKT);
  x.nsteps = static_cast<int>(s1 - s0);
  x.rev = 0;
  return true;
}

template <int FMT, bool ZP, bool UB>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    dw_pair_kernel(const __grid_constant__ CUtensorMap tm_dy, const __grid_constant__ CUtensorMap tm_x,
                   const __grid_constant__ CUtensorMap tm_at, const __grid_constant__ CUtensorMap tm_ath,
                   const __grid_constant__ CUtensorMap tm_phi, const __grid_constant__ CUtensorMap tm_b,
                   const __grid_constant__ CUtensorMap tm_bh, const DwArgs args) {
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
  constexpr bool PACKED = FMT == FMT_I4;
  constexpr bool P16 = fmt_16bit(FMT);   // base read from global memory by the epilogue
  constexpr int BN = 256;
  const uint32_t rbox = static_cast<uint32_t>(args.r16) * 128u;   // bytes of one r16-row x 64-col box
  const uint32_t hbox = rbox / 2;                                  // bytes of one r16/2-row x 64-col box
  const int ni128 = 2 * args.ni;                                   // 128-row blocks

  if (threadIdx.x == 0) {
    abort_s = 0;
    for (int s = 0; s < NS; ++s) {
      mbar_init(bar(BAR_FULL + s), 1);
      mbar_init(bar(BAR_EMPTY + s), 1);
    }
    mbar_init(bar(BAR_EFFULL), 1);
    mbar_init(bar(BAR_EFEMPTY), 1);
    mbar_init(bar(BAR_ECFULL), 1);
    mbar_init(bar(BAR_ECEMPTY), 1);
    mbar_init(bar(BAR_PFULL), 1);
    mbar_init(bar(BAR_ACCFULL), 1);
    mbar_init(bar(BAR_ACCEMPTY), NUM_EPI_WARPS);
    mbar_init(bar(BAR_LFULL), 1);
    mbar_init(bar(BAR_DUFULL), NUM_EPI_WARPS);
    mbar_init(bar(BAR_DBFULL), 1);
    mbar_init(bar(BAR_DRAIN), 1);
    mbar_init(bar(BAR_DRAIN_E), 1);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc_pair(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();   // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};
  const uint32_t sig_src = smem_u32(&sig_buf[0]);
  const uint32_t sig_dst_leader = map_shared_rank(smem_u32(&sig_buf[4]), 0);

  if (warp == 0) {
    // ---------------------------------------- epilogue operands (per unit/chunk)
    if (lane == 0) {
      prefetch_tensormap(&tm_at);
      prefetch_tensormap(&tm_ath);
      prefetch_tensormap(&tm_b);
      prefetch_tensormap(&tm_bh);
      if (!P16) prefetch_tensormap(&tm_phi);
      const uint32_t half = static_cast<uint32_t>(args.r16 / 2);   // this CTA's rank rows of the halves
      uint32_t it = 0, cc = 0;
      bool ok = true;
      WorkIter wi = work_begin(args, pair);
      Unit w;
      while (ok && work_next(wi, args, pair, npairs, w)) {
        if (args.sched.tail && w.sp == 0) {   // the reduction reads which slots hold data
          const int64_t tile2 = w.ib + static_cast<int64_t>(args.ni) * w.jt;
          args.tile_segs[(2 * w.ib + static_cast<int>(rank)) + static_cast<int64_t>(ni128) * w.jt] =
              dw_tile_segments(tile2, args.sched);
        }
        const int i_pair = w.ib * 256, i_own = i_pair + static_cast<int>(rank) * 128;
        if (!(ok = wait_spin_bounded(bar(BAR_EFEMPTY), (it & 1u) ^ 1u, ctl, 2))) break;
        if (leader) mbar_arrive_expect_tx(bar(BAR_EFFULL), 2u * (2u * rbox + 4u * hbox));
        tma_load_2d_pair(smem + OFF_AT, &tm_at, i_own, 0, lbar(BAR_EFFULL));
        tma_load_2d_pair(smem + OFF_AT + rbox, &tm_at, i_own + 64, 0, lbar(BAR_EFFULL));
#pragma unroll
        for (int hi = 0; hi < 2; ++hi) {   // rows i of CTA hi, this CTA's rank half
          const uint32_t dst = smem + OFF_ATH + hi * 2u * hbox;
          tma_load_2d_pair(dst, &tm_ath, i_pair + 128 * hi, static_cast<int>(rank * half), lbar(BAR_EFFULL));
          tma_load_2d_pair(dst + hbox, &tm_ath, i_pair + 128 * hi + 64, static_cast<int>(rank * half),
                           lbar(BAR_EFFULL));
        }
        ++it;
        for (int c = 0; c < 2; ++c) {
          if (!(ok = wait_spin_bounded(bar(BAR_ECEMPTY), (cc & 1u) ^ 1u, ctl, 3))) break;
          const int j0 = w.jt * BN + 128 * c;
          if (!P16) {
            mbar_arrive_expect_tx(bar(BAR_PFULL), PACKED ? 8192u : 16384u);
            tma_load_2d(smem + OFF_PHI, &tm_phi, PACKED ? j0 / 2 : j0, i_own, bar(BAR_PFULL));
          }
          if (leader) mbar_arrive_expect_tx(bar(BAR_ECFULL), 2u * (rbox + 2u * hbox));
          tma_load_2d_pair(smem + OFF_BPL, &tm_b, j0 + 64 * static_cast<int>(rank), 0, lbar(BAR_ECFULL));
          tma_load_2d_pair(smem + OFF_BPA, &tm_bh, j0, static_cast<int>(rank * half), lbar(BAR_ECFULL));
          tma_load_2d_pair(smem + OFF_BPA + hbox, &tm_bh, j0 + 64, static_cast<int>(rank * half), lbar(BAR_ECFULL));
          ++cc;
        }
      }
      // the copies that complete on this CTA's own barrier land before the CTA ends (those on
      // the leader's barriers are all waited for by its MMA thread)
      if (!P16 && cc > 0) drain_wait(bar(BAR_PFULL), (cc - 1) & 1u, args.timeout_ns);
    }
  } else if (warp >= FIRST_LOADER && warp < FIRST_LOADER + NUM_LOADERS) {
    // ------------------------------------------------ pipeline stage loaders
    // Loader b issues box b of every stage (boxes 0-1: this CTA's dY columns i, boxes 2-3: its X
    // columns j): one warp's copies are handled one after another, so a stage's four boxes are
    // fetched by four warps at once.  Loader 0 of the leader announces the stage's bytes.
    const int b = warp - FIRST_LOADER;
    if (lane == 0) {
      if (b < 2) prefetch_tensormap(&tm_dy);
      else prefetch_tensormap(&tm_x);
      uint32_t g = 0;
      bool ok = true;
      WorkIter wi = work_begin(args, pair);
      Unit w;
      while (ok && work_next(wi, args, pair, npairs, w)) {
        const int i_own = w.ib * 256 + static_cast<int>(rank) * 128;
        const int j_own = w.jt * BN + static_cast<int>(rank) * 128;
        for (int step = 0; step < w.nsteps; ++step, ++g) {
          const uint32_t s = g % NS, ph = (g / NS) & 1u;
          if (!(ok = wait_spin_bounded(bar(BAR_EMPTY + s), ph ^ 1u, ctl, 1))) break;
          const uint32_t st = smem + OFF_STAGES + s * STAGE_BYTES;
          const uint32_t fb = lbar(BAR_FULL + s);
          if (b == 0 && leader) mbar_arrive_expect_tx(bar(BAR_FULL + s), 2u * STAGE_BYTES);
          const int tok = w.t0 + (w.rev ? w.nsteps - 1 - step : step) * BKT;
          if (b < 2) tma_load_2d_pair(st + b * BOX_BYTES, &tm_dy, i_own + 64 * b, tok, fb);
          else tma_load_2d_pair(st + STAGE_DY + (b - 2) * BOX_BYTES, &tm_x, j_own + 64 * (b - 2), tok, fb);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------ MMA issuer (the leader's)
    if (lane == 0 && leader) {
      const uint32_t idesc_g = make_idesc_bf16(256, BN, 1, 1);
      const uint64_t d_dy0 = make_sdesc(smem + OFF_STAGES, BOX_BYTES, 1024, SWZ_128B);
      const uint64_t d_x0 = make_sdesc(smem + OFF_STAGES + STAGE_DY, BOX_BYTES, 1024, SWZ_128B);
      const uint32_t b_full = bar(BAR_FULL);
      uint32_t it = 0;
      uint32_t s = 0, ph = 0;   // stage and phase of the global step
      bool ok = true;
      WorkIter wi = work_begin(args, pair);
      Unit w;
      while (ok && work_next(wi, args, pair, npairs, w)) {
        if (!(ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 4))) break;
        tc_fence_after();
        for (int step = 0; step < w.nsteps; ++step) {
          if (!(ok = wait_spin_bounded(b_full + 8u * s, ph, ctl, 5))) break;
          tc_fence_after();
          const uint64_t a = d_dy0 + s * (STAGE_BYTES >> 4), b = d_x0 + s * (STAGE_BYTES >> 4);
#pragma unroll
          for (int kq = 0; kq < BKT / 16; ++kq)   // 16-token K steps: 16 rows of 128 bytes
            mma_bf16_pair(tmem + COL_G, a + 128 * kq, b + 128 * kq, idesc_g, (step > 0 || kq > 0) ? 1u : 0u);
          mma_commit_pair(bar(BAR_EMPTY + s));
          if (++s == NS) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit_pair(bar(BAR_ACCFULL));
        ++it;
      }
      // the peer's last drain report lands before the CTAs end
      if (ok) ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 14);
      mma_commit_pair_self(bar(BAR_DRAIN));
      drain_wait(bar(BAR_DRAIN), 0, args.timeout_ns);
    }
  } else if (warp == EPI_MMA_WARP) {
    // -------------------------------------------- epilogue MMA issuer (the leader's)
    // The low-rank tiles and the adapter contractions of every unit, issued by a thread of their
    // own: the next unit's main loop (warp 1) starts as soon as the epilogue has read G, and
    // the first chunk's low-rank tile is computed while the unit's main loop still runs.
    if (lane == 0 && leader) {
      const uint32_t idesc_l = make_idesc_bf16(256, 128, 1, 1);
      const uint32_t idesc_da = make_idesc_bf16(256, args.r16, 0, 0);
      const uint32_t idesc_db = make_idesc_bf16(256, args.r16, 1, 0);
      const int lsteps = args.r16 / 16;
      uint32_t it = 0, cc = 0;
      bool ok = true;
      WorkIter wi = work_begin(args, pair);
      Unit w;
      while (ok && work_next(wi, args, pair, npairs, w)) {
        if (!(ok = wait_spin_bounded(bar(BAR_EFFULL), it & 1u, ctl, 6))) break;
        for (int c = 0; c < 2; ++c) {
          if (!(ok = wait_spin_bounded(bar(BAR_ECFULL), cc & 1u, ctl, 7))) break;
          tc_fence_after();
          // L = A (rows i) * B (the chunk's columns j): both operands MN-major, 16 rank rows
          // (two 8-row groups) per K step; each CTA supplies its 64 columns of B.  Both CTAs'
          // epilogue warps read the previous chunk's L before they reported its dU (DUFULL).
          for (int ks = 0; ks < lsteps; ++ks) {
            const uint64_t ad = make_sdesc(smem + OFF_AT + 2048u * ks, rbox, 1024, SWZ_128B);
            const uint64_t bd = make_sdesc(smem + OFF_BPL + 2048u * ks, rbox, 1024, SWZ_128B);
            mma_bf16_pair(tmem + COL_L, ad, bd, idesc_l, ks > 0 ? 1u : 0u);
          }
          mma_commit_pair(bar(BAR_LFULL));
          if (!(ok = wait_spin_bounded(bar(BAR_DUFULL), cc & 1u, ctl, 8))) break;
          tc_fence_after();
          // dA (+)= dU * B_chunk^T : M = 256 rows i, N = r16 (half per CTA), K = 128 columns j
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t ad = make_sdesc(smem + OFF_DU + 16384u * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
            const uint64_t bd = make_sdesc(smem + OFF_BPA + hbox * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
            mma_bf16_pair(tmem + COL_DA, ad, bd, idesc_da, (c > 0 || ks > 0) ? 1u : 0u);
          }
          // dB^T partials = dU^T * A : M = 128 columns j per CTA (dU read MN-major), N = r16
          // (half per CTA), K = the 128 rows of CTA hi, written into CTA hi's lanes only
#pragma unroll
          for (int hi = 0; hi < 2; ++hi) {
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              const uint64_t ad = make_sdesc(smem + OFF_DU + 2048u * ks, 16384, 1024, SWZ_128B);
              const uint64_t bd = make_sdesc(smem + OFF_ATH + hi * 2u * hbox + hbox * (ks >> 2) + 32u * (ks & 3), 16,
                                             1024, SWZ_128B);
              mma_bf16_pair_half(tmem + COL_DBT, ad, bd, idesc_db, ks > 0 ? 1u : 0u, hi);
            }
          }
          mma_commit_pair(bar(BAR_DBFULL));
          mma_commit_pair(bar(BAR_ECEMPTY));
          ++cc;
        }
        if (!ok) break;
        mma_commit_pair(bar(BAR_EFEMPTY));
        ++it;
      }
      mma_commit_pair_self(bar(BAR_DRAIN_E));
      drain_wait(bar(BAR_DRAIN_E), 0, args.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int pw = warp - 2;
    const int q = warp & 3;
    const int h = pw >> 2;
    const int row = q * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const QuantParams qp = args.q;
    const uint32_t lr2 = pack_rn_bf16x2(qp.lr_scale, qp.lr_scale);   // exact: a power of two when UB
    const int nb = args.k / 128;
    const float gscale = args.s_x != nullptr ? *args.s_x : 1.0f;
    const int half_cols = args.r16 / 2;   // dA / dB^T columns read by this warp half
    // A warp's event on a leader barrier: the leader's warps arrive (warp 0 also announces
    // the peer's signal bytes), the peer's warps send their signal.
    auto report = [&](int b) {
      if (leader) {
        if (pw == 0) mbar_arrive_expect_tx(bar(b), SIG_TX);
        else mbar_arrive(bar(b));
      } else {
        signal_remote16(sig_dst_leader, sig_src, lbar(b));
      }
    };
    uint32_t it = 0, cc = 0;
    bool ok = true;
    WorkIter wi = work_begin(args, pair);
    Unit w;
    while (ok && work_next(wi, args, pair, npairs, w)) {
      const int ib128 = 2 * w.ib + static_cast<int>(rank);
      const int i_g = ib128 * 128 + row;
      ok = wait_bounded(bar(BAR_ACCFULL), it & 1u, ctl, 9);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      for (int c = 0; c < 2; ++c) {
        const int j0 = w.jt * BN + 128 * c;
        // 16-bit base: this thread's 2 x 32 values of row i_g (columns 64 h .. 64 h + 63)
        uint4 g16[8];
        if (P16) {
          const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(args.phi) +
                                                            static_cast<int64_t>(i_g) * args.k + j0 + 64 * h);
#pragma unroll
          for (int e = 0; e < 8; ++e) g16[e] = __ldg(src + e);
        }
        const float s_i = args.s_ld ? args.s[static_cast<int64_t>(i_g) * args.s_ld + j0 / args.group_size]
                                    : args.s[i_g];
        const float z_i = !ZP         ? 0.0f
                          : args.s_ld ? args.zero[static_cast<int64_t>(i_g) * args.s_ld + j0 / args.group_size]
                                      : args.zero[i_g];
        ok = P16 || wait_bounded(bar(BAR_PFULL), cc & 1u, ctl, 10);
        ok = ok && wait_bounded(bar(BAR_LFULL), cc & 1u, ctl, 11);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
        // Packed fp32x2 arithmetic per pair of columns, as in the one-SM kernel.
        const float gs_i = gscale * s_i;
        const float code_n = __fmaf_rn(qp.lo, qp.inv2f, -qp.magic_c);   // n and p as exact floats
        const float code_p = __fmaf_rn(qp.hi, qp.inv2f, -qp.magic_c);
        float2 ds2 = make_float2(0.0f, 0.0f);
#pragma unroll 1
        for (int p = 0; p < 2; ++p) {
          const int jl = 64 * h + 32 * p;   // column within the chunk
          float G[32], Lv[32], v[32];
          tmem_ld32(tmem + lane_off + COL_G + 128 * c + jl, G);
          tmem_ld32(tmem + lane_off + COL_L + jl, Lv);
          tmem_ld_wait();
          uint32_t raw[16];
          if (PACKED) {
            const uint4 r0 = ld_shared_v4(smem + OFF_PHI + swz_offset(row, jl / 32, 64));
            raw[0] = r0.x, raw[1] = r0.y, raw[2] = r0.z, raw[3] = r0.w;
            decode16<FMT>(raw, v);
            decode16<FMT>(raw + 2, v + 16);
          } else if (P16) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const uint4 r0 = g16[4 * p + e];
              raw[4 * e] = r0.x, raw[4 * e + 1] = r0.y, raw[4 * e + 2] = r0.z, raw[4 * e + 3] = r0.w;
            }
            decode16<FMT>(raw, v);
            decode16<FMT>(raw + 8, v + 16);
          } else {
            const uint4 r0 = ld_shared_v4(smem + OFF_PHI + swz_offset(row, jl / 16, 128));
            const uint4 r1 = ld_shared_v4(smem + OFF_PHI + swz_offset(row, jl / 16 + 1, 128));
            raw[0] = r0.x, raw[1] = r0.y, raw[2] = r0.z, raw[3] = r0.w;
            raw[4] = r1.x, raw[5] = r1.y, raw[6] = r1.z, raw[7] = r1.w;
            decode16<FMT>(raw, v);
            decode16<FMT>(raw + 4, v + 16);
          }
          uint32_t du[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const float2 g2 = make_float2(G[2 * e], G[2 * e + 1]);
            const float2 v2 = make_float2(v[2 * e], v[2 * e + 1]);
            const float2 u2 = UB ? u_bf16x2(Lv[2 * e], Lv[2 * e + 1], v2.x, v2.y, lr2)
                                 : __ffma2_rn(make_float2(Lv[2 * e], Lv[2 * e + 1]),
                                              make_float2(qp.lr_scale, qp.lr_scale), v2);
            const float2 t2 = __fadd2_rn(u2, make_float2(qp.magic, qp.magic));
            const float2 cu = __ffma2_rn(t2, make_float2(qp.inv2f, qp.inv2f), make_float2(-qp.magic_c, -qp.magic_c));
            const float2 cl = make_float2(fminf(fmaxf(cu.x, code_n), code_p), fminf(fmaxf(cu.y, code_n), code_p));
            ds2 = __ffma2_rn(g2, ZP ? __fadd2_rn(cl, make_float2(-z_i, -z_i)) : cl, ds2);
            const float2 gs = __fmul2_rn(g2, make_float2(gs_i, gs_i));
            du[e] = pack_rn_bf16x2(cl.x == cu.x ? gs.x : 0.0f, cl.y == cu.y ? gs.y : 0.0f);
          }
          const uint32_t dub = smem + OFF_DU + 16384u * h;
#pragma unroll
          for (int wq = 0; wq < 4; ++wq)
            st_shared_v4(dub + swz_offset(row, 4 * p + wq, 128), du[4 * wq], du[4 * wq + 1], du[4 * wq + 2],
                         du[4 * wq + 3]);
        }
        if (c == 1) {
          // Last read of G for this unit: hand the accumulator to the next unit's main loop,
          // which then overlaps the adapter contractions and partial stores below.
          tc_fence_before();
          __syncwarp();
          if (lane == 0) report(BAR_ACCEMPTY);
        }
        const float ds_acc = (ds2.x + ds2.y) * gscale;
        args.ds_part[(static_cast<int64_t>(w.sp * 2 + h) * args.m + i_g) * nb + j0 / 128] = ds_acc;
        tc_fence_before();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) report(BAR_DUFULL);
        ok = wait_bounded(bar(BAR_DBFULL), cc & 1u, ctl, 12);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
        // dB^T partial of this CTA's rows: lanes = columns j of the chunk, TMEM columns = ranks
        {
          float* dst = args.dB_part + static_cast<int64_t>(ib128 * args.nsplit + w.sp) * args.r * args.k + j0 + row;
          for (int c8 = 0; c8 < half_cols; c8 += 8) {
            float vv[8];
            tmem_ld8(tmem + lane_off + COL_DBT + h * half_cols + c8, vv);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int t = h * half_cols + c8 + e;
              if (t < args.r) dst[static_cast<int64_t>(t) * args.k] = vv[e];
            }
          }
        }
        if (c == 1) {
          float* dst = args.dA_part + (static_cast<int64_t>(w.jt * args.nsplit + w.sp) * args.m + i_g) * args.r;
          for (int c8 = 0; c8 < half_cols; c8 += 8) {
            float vv[8];
            tmem_ld8(tmem + lane_off + COL_DA + h * half_cols + c8, vv);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int t = h * half_cols + c8 + e;
              if (t < args.r) dst[t] = vv[e];
            }
          }
        }
        ++cc;
      }
      if (!ok) break;
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

struct PairMaps {
  const CUtensorMap *dy, *x, *at, *ath, *phi, *b, *bh;
};

template <int FMT, bool ZP, bool UB>
cudaError_t launch_pair_one(const PairMaps& m, const DwArgs& args, int npairs, cudaStream_t stream) {
  static bool configured[kMaxDevices] = {};
  const void* fn = reinterpret_cast<const void*>(dw_pair_kernel<FMT, ZP, UB>);
  cudaError_t e = ensure_smem_attr(fn, static_cast<int>(SMEM_BYTES), configured);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(static_cast<unsigned>(2 * npairs), 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, dw_pair_kernel<FMT, ZP, UB>, *m.dy, *m.x, *m.at, *m.ath, *m.phi, *m.b, *m.bh, args);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int FMT>
cudaError_t launch_pair_fmt(const PairMaps& m, const DwArgs& args, int npairs, cudaStream_t stream) {
  if (args.u_bf16) {   // bf16 pre-round value: no zero offsets, bases exact in bf16
    if (FMT == FMT_F16 || args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_pair_one<FMT == FMT_F16 ? FMT_Q8 : FMT, false, true>(m, args, npairs, stream);
  }
  if (fmt_float(FMT)) {
    if (args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_pair_one<FMT, false, false>(m, args, npairs, stream);
  }
  return args.zero != nullptr ? launch_pair_one<FMT, true, false>(m, args, npairs, stream)
                              : launch_pair_one<FMT, false, false>(m, args, npairs, stream);
}

}  // namespace

int dw_pair_max_pairs() {
  static int cache[kMaxDevices] = {};
  static bool configured[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  if (cache[dev] > 0) return cache[dev];
  const void* fn = reinterpret_cast<const void*>(dw_pair_kernel<FMT_Q8, false, false>);
  if (ensure_smem_attr(fn, static_cast<int>(SMEM_BYTES), configured) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(NUM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, dw_pair_kernel<FMT_Q8, false, false>, &cfg) != cudaSuccess) return 0;
  cache[dev] = n;
  return n;
}

cudaError_t launch_dw_pair(int fmt, const CUtensorMap& tm_dy, const CUtensorMap& tm_x, const CUtensorMap& tm_at,
                           const CUtensorMap& tm_ath, const CUtensorMap& tm_phi, const CUtensorMap& tm_b,
                           const CUtensorMap& tm_bh, const DwArgs& args, int npairs, cudaStream_t stream) {
  if (npairs < 1 || args.codes_base || args.nchunks != 2 || args.r16 < 16 || args.r16 > 64 || (args.r16 & 15) ||
      args.m % 256 || args.k % 256 || args.ni != args.m / 256 || args.nj != args.k / 256)
    return cudaErrorInvalidValue;
  if (fmt_16bit(fmt) && (args.phi == nullptr || (reinterpret_cast<uintptr_t>(args.phi) & 15u)))
    return cudaErrorInvalidValue;
  const PairMaps m{&tm_dy, &tm_x, &tm_at, &tm_ath, &tm_phi, &tm_b, &tm_bh};
  switch (fmt) {
    case FMT_Q8: return launch_pair_fmt<FMT_Q8>(m, args, npairs, stream);
    case FMT_I4: return launch_pair_fmt<FMT_I4>(m, args, npairs, stream);
    case FMT_BF16: return launch_pair_fmt<FMT_BF16>(m, args, npairs, stream);
    case FMT_F16: return launch_pair_fmt<FMT_F16>(m, args, npairs, stream);
    case FMT_E4M3: return launch_pair_fmt<FMT_E4M3>(m, args, npairs, stream);
    case FMT_E5M2: return launch_pair_fmt<FMT_E5M2>(m, args, npairs, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lrqat
