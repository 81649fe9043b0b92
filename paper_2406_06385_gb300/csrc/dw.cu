// Fused weight-gradient kernel of the LR-QAT layer.  For a tile of 128 weight
// rows i x (128 or 256) columns j and a range of tokens it computes
//   G = dY^T X_hat                 (tcgen05, fp32 accumulator in TMEM, never stored)
// and, in the epilogue, the straight-through gradients of Eq. 8:
//   u = phi^{-1}(Phi0) + (alpha/r) A B   (low-rank tile by tcgen05, recomputed)
//   M = 1[n <= round(u) <= p],  c = clip(round(u), n, p)
//   dU = G * s * M  -> bf16 in shared memory
//   dA_partial = dU B^T,  dB^T_partial = dU^T A   (tcgen05, N = r rounded to 16)
//   ds_partial = sum_j G * c
// The partials of dA, dB and ds are reduced deterministically by a later kernel.
//
// A 16-bit base (BF16/FP16 storage) would need a 32 KB chunk in shared memory, which
// the pipeline leaves no room for: the epilogue threads read it from global memory
// instead (each thread 64 contiguous bytes of its own row per half chunk, issued
// before the waits of the chunk so that the latency overlaps them).
//
// Roles (416 threads): warp 0 loads the epilogue operands, warp 1 issues tcgen05
// MMAs and owns TMEM, warps 2..9 run the epilogue, warps 10..12 fill the pipeline
// stages with TMA.  Work units (row block, column tile, token split) are
// distributed persistently over the CTAs.
//
// Ranks above 64 (NL): the base holds the unclipped codes round(u), low-rank term
// included (the tensor-core code pass writes them once per call), so no low-rank tile
// is computed, and the tiles are 128 columns wide.  The adapter contractions run in
// rounds of 64 rank indices: per round the slices A^T[64 ranks, 128 rows] and B[64
// ranks, 128 columns] land in the epilogue buffers, tcgen05 computes that round's 64
// columns of dU B^T and dU^T A into one of two TMEM buffers, and the epilogue warps
// write them out while the next round runs in the other buffer.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int NS = 6;
constexpr int BKT = 32;                        // tokens per pipeline stage
constexpr int NUM_EPI_WARPS = 8;
// TMA instructions issued by one warp are processed one after another, so the
// pipeline stages are filled round-robin by NUM_LOADERS warps (one box per lane);
// warp 0 loads the per-unit epilogue operands.
constexpr int NUM_LOADERS = 3;
constexpr int FIRST_LOADER = 2 + NUM_EPI_WARPS;
constexpr int NUM_THREADS = 32 * (FIRST_LOADER + NUM_LOADERS);

constexpr uint32_t BOX_BYTES = 64 * 32 * 2;    // one 64-column x 32-token bf16 box (SW128)
constexpr uint32_t STAGE_DY = 2 * BOX_BYTES;   // 128 rows i
constexpr uint32_t STAGE_BYTES = STAGE_DY + 4 * BOX_BYTES;   // + up to 256 columns j
constexpr uint32_t OFF_STAGES = 0;
// A^T [r16 rows t, 128 columns i] (2 boxes of 64 i) serves as the MN-major A operand of
// the low-rank tile and the K-major B operand of dU^T A; B (padded) [r16 rows t, 128
// columns j] serves as the MN-major B operand of the low-rank tile and the K-major B
// operand of dU B^T.
constexpr uint32_t OFF_AT = OFF_STAGES + NS * STAGE_BYTES;     // A^T: 2 boxes of r16 rows x 64 cols
constexpr uint32_t OFF_PHI = OFF_AT + 16384;                   // Phi0 chunk 128 x 128 (packed: 128 x 64 B)
constexpr uint32_t OFF_BP = OFF_PHI + 16384;                   // B (padded) chunk: 2 boxes of r16 rows x 64 cols
constexpr uint32_t OFF_DU = OFF_BP + 16384;                    // dU chunk: 2 atom columns of 128 rows x 128 B
constexpr uint32_t SMEM_TILES = OFF_DU + 32768;
constexpr uint32_t SMEM_BYTES = SMEM_TILES + 1024;
static_assert(SMEM_BYTES <= 232448, "shared memory budget");

constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_G = 0;      // 256 columns
constexpr uint32_t COL_L = 256;    // 128 columns
constexpr uint32_t COL_DA = 384;   // up to 64 columns
constexpr uint32_t COL_DBT = 448;  // up to 64 columns
// NL: two buffers of a round's contractions, dA at COL_NL + 128 b, dB^T 64 columns further
constexpr uint32_t COL_NL = 256;
constexpr uint32_t NL_BOX = 64 * 128;   // one 64-rank-row x 64-column bf16 box

constexpr int BAR_FULL = 0;
constexpr int BAR_EMPTY = BAR_FULL + NS;
constexpr int BAR_EFFULL = BAR_EMPTY + NS;
constexpr int BAR_EFEMPTY = BAR_EFFULL + 1;
constexpr int BAR_ECFULL = BAR_EFEMPTY + 1;
constexpr int BAR_ECEMPTY = BAR_ECFULL + 1;
constexpr int BAR_ACCFULL = BAR_ECEMPTY + 1;
constexpr int BAR_ACCEMPTY = BAR_ACCFULL + 1;
constexpr int BAR_LFULL = BAR_ACCEMPTY + 1;
constexpr int BAR_DUFULL = BAR_LFULL + 1;
constexpr int BAR_DBFULL = BAR_DUFULL + 1;
constexpr int BAR_DRAIN = BAR_DBFULL + 1;
// NL: the second buffer's contractions done, and each buffer read by the epilogue
constexpr int BAR_DBFULL1 = BAR_DRAIN + 1;
constexpr int BAR_DRAINED = BAR_DBFULL1 + 1;   // two barriers
constexpr int NUM_BARS = BAR_DRAINED + 2;

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) break;
  }
}

struct Unit {
  int ib, jt, sp, t0, nsteps;
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
  return x;
}

// Whole tile number u (u < full_tiles, in processing order) of the tail schedule.  The whole
// tiles are the natural indices ib + ni jt < full_tiles; they are taken in groups of
// kColGroup column tiles with the column tile varying fastest, so that a wave of CTAs covers
// about (CTAs / kColGroup) row blocks x kColGroup column tiles: a rectangle of dY and X
// columns rather than every row block (all of dY) per wave.  The part of the prefix that does
// not fill a whole group keeps the natural order.
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

// This CTA's units (equal token splits, taken round robin), or (tail schedule) its whole
// tiles of the full waves followed by its one part of a tail tile (slot = part index).
struct WorkIter {
  int64_t u;      // next unit, or next whole tile
  bool tail;      // the tail part is still to come
};

__device__ __forceinline__ WorkIter work_begin(const DwArgs& a) {
  return {static_cast<int64_t>(blockIdx.x), a.sched.tail != 0 && blockIdx.x < a.sched.tail_grid};
}

__device__ __forceinline__ bool work_next(WorkIter& it, const DwArgs& a, Unit& x) {
  if (!a.sched.tail) {
    if (it.u >= a.num_units) return false;
    x = decode_unit(static_cast<int>(it.u), a);
    it.u += gridDim.x;
    return true;
  }
  if (it.u < a.sched.full_tiles) {
    dw_whole_tile(it.u, a.ni, a.sched.full_tiles, x.ib, x.jt);
    x.sp = 0;
    x.t0 = 0;
    x.nsteps = static_cast<int>(a.sched.tsteps);
    it.u += gridDim.x;
    return true;
  }
  if (!it.tail) return false;
  it.tail = false;
  int64_t t;
  int j, q;
  dw_tail_part(blockIdx.x, a.sched, t, j, q);
  const int64_t tile = a.sched.full_tiles + t;
  const int64_t s0 = j * a.sched.tsteps / q, s1 = (j + 1) * a.sched.tsteps / q;
  x.ib = static_cast<int>(tile % a.ni);
  x.jt = static_cast<int>(tile / a.ni);
  x.sp = j;
  x.t0 = static_cast<int>(s0 * BKT);
  x.nsteps = static_cast<int>(s1 - s0);
  return true;
}

// UB: pre-round value in bf16 (u_bf16x2) instead of one fp32 FMA.
// NL: the base holds the unclipped codes (FMT_Q8, 0 fraction bits), no low-rank tile,
// 128-column tiles, adapter contractions in rounds of 64 ranks.
template <int FMT, bool ZP, bool UB, bool NL>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    dw_kernel(const __grid_constant__ CUtensorMap tm_dy, const __grid_constant__ CUtensorMap tm_x,
              const __grid_constant__ CUtensorMap tm_at, const __grid_constant__ CUtensorMap tm_phi,
              const __grid_constant__ CUtensorMap tm_b, const DwArgs args) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[NUM_BARS];
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int abort_s;

  const uint32_t smem = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  constexpr bool PACKED = FMT == FMT_I4;
  constexpr bool P16 = fmt_16bit(FMT);   // base read from global memory by the epilogue
  const int BN = 128 * args.nchunks;
  const uint32_t rbox = static_cast<uint32_t>(args.r16) * 128u;   // bytes of one r16-row x 64-col box

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
    mbar_init(bar(BAR_ACCFULL), 1);
    mbar_init(bar(BAR_ACCEMPTY), NUM_EPI_WARPS);
    mbar_init(bar(BAR_LFULL), 1);
    mbar_init(bar(BAR_DUFULL), NUM_EPI_WARPS);
    mbar_init(bar(BAR_DBFULL), 1);
    mbar_init(bar(BAR_DRAIN), 1);
    mbar_init(bar(BAR_DBFULL1), 1);
    mbar_init(bar(BAR_DRAINED), NUM_EPI_WARPS);
    mbar_init(bar(BAR_DRAINED + 1), NUM_EPI_WARPS);
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};

  if (warp == 0) {
    // ---------------------------------------- epilogue operands (per unit/chunk)
    if (NL && lane == 0) {
      // the unit's code chunk, then its rank rounds (A^T and B slices of 64 ranks)
      const int nrc = (args.r16 + 63) / 64;
      uint32_t it = 0, cc = 0;
      bool ok = true;
      WorkIter wi = work_begin(args);
      Unit w;
      while (ok && work_next(wi, args, w)) {
        if (args.sched.tail && w.sp == 0) {
          const int64_t tile = w.ib + static_cast<int64_t>(args.ni) * w.jt;
          args.tile_segs[tile] = dw_tile_segments(tile, args.sched);
        }
        if (!(ok = wait_spin_bounded(bar(BAR_ECEMPTY), (cc & 1u) ^ 1u, ctl, 3))) break;
        const int j0 = w.jt * 128;
        mbar_arrive_expect_tx(bar(BAR_ECFULL), 16384u);
        tma_load_2d(smem + OFF_PHI, &tm_phi, j0, w.ib * 128, bar(BAR_ECFULL));
        ++cc;
        for (int rc = 0; rc < nrc; ++rc) {
          if (!(ok = wait_spin_bounded(bar(BAR_EFEMPTY), (it & 1u) ^ 1u, ctl, 2))) break;
          mbar_arrive_expect_tx(bar(BAR_EFFULL), 4u * NL_BOX);
          tma_load_2d(smem + OFF_AT, &tm_at, w.ib * 128, 64 * rc, bar(BAR_EFFULL));
          tma_load_2d(smem + OFF_AT + NL_BOX, &tm_at, w.ib * 128 + 64, 64 * rc, bar(BAR_EFFULL));
          tma_load_2d(smem + OFF_BP, &tm_b, j0, 64 * rc, bar(BAR_EFFULL));
          tma_load_2d(smem + OFF_BP + NL_BOX, &tm_b, j0 + 64, 64 * rc, bar(BAR_EFFULL));
          ++it;
        }
      }
      if (it > 0) drain_wait(bar(BAR_EFFULL), (it - 1) & 1u, args.timeout_ns);
      if (cc > 0) drain_wait(bar(BAR_ECFULL), (cc - 1) & 1u, args.timeout_ns);
    } else if (lane == 0) {
      const uint32_t ef_tx = 2u * rbox;
      const uint32_t ec_tx = (P16 ? 0u : PACKED ? 8192u : 16384u) + 2u * rbox;
      uint32_t it = 0, cc = 0;
      bool ok = true;
      WorkIter wi = work_begin(args);
      Unit w;
      while (ok && work_next(wi, args, w)) {
        if (args.sched.tail && w.sp == 0) {   // the reduction reads which slots hold data
          const int64_t tile = w.ib + static_cast<int64_t>(args.ni) * w.jt;
          args.tile_segs[tile] = dw_tile_segments(tile, args.sched);
        }
        if (!(ok = wait_spin_bounded(bar(BAR_EFEMPTY), (it & 1u) ^ 1u, ctl, 2))) break;
        mbar_arrive_expect_tx(bar(BAR_EFFULL), ef_tx);
        tma_load_2d(smem + OFF_AT, &tm_at, w.ib * 128, 0, bar(BAR_EFFULL));
        tma_load_2d(smem + OFF_AT + rbox, &tm_at, w.ib * 128 + 64, 0, bar(BAR_EFFULL));
        ++it;
        for (int c = 0; c < args.nchunks; ++c) {
          if (!(ok = wait_spin_bounded(bar(BAR_ECEMPTY), (cc & 1u) ^ 1u, ctl, 3))) break;
          const int j0 = w.jt * BN + 128 * c;
          mbar_arrive_expect_tx(bar(BAR_ECFULL), ec_tx);
          if (!P16) tma_load_2d(smem + OFF_PHI, &tm_phi, PACKED ? j0 / 2 : j0, w.ib * 128, bar(BAR_ECFULL));
          tma_load_2d(smem + OFF_BP, &tm_b, j0, 0, bar(BAR_ECFULL));
          tma_load_2d(smem + OFF_BP + rbox, &tm_b, j0 + 64, 0, bar(BAR_ECFULL));
          ++cc;
        }
      }
      if (it > 0) drain_wait(bar(BAR_EFFULL), (it - 1) & 1u, args.timeout_ns);
      if (cc > 0) drain_wait(bar(BAR_ECFULL), (cc - 1) & 1u, args.timeout_ns);
    }
  } else if (warp >= FIRST_LOADER) {
    // ------------------------------------------------ pipeline stage loaders
    // Loader t fills the global steps g = t, t + NUM_LOADERS, ...; lane b issues box b
    // (boxes 0-1: dY columns i, boxes 2..: X columns j).
    const uint32_t t = warp - FIRST_LOADER;
    if (lane == 0) {
      prefetch_tensormap(&tm_dy);
      prefetch_tensormap(&tm_x);
    }
    const uint32_t stage_tx = STAGE_DY + 2u * args.nchunks * BOX_BYTES;
    const int nbox = 2 + 2 * args.nchunks;
    uint32_t g = 0, last_g = 0xffffffffu;
    bool ok = true;
    WorkIter wi = work_begin(args);
    Unit w;
    while (ok && work_next(wi, args, w)) {
      for (int step = 0; step < w.nsteps; ++step, ++g) {
        if (g % NUM_LOADERS != t) continue;
        const uint32_t s = g % NS, ph = (g / NS) & 1u;
        if (lane == 0) ok = wait_spin_bounded(bar(BAR_EMPTY + s), ph ^ 1u, ctl, 1);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        const uint32_t st = smem + OFF_STAGES + s * STAGE_BYTES;
        const uint32_t fb = bar(BAR_FULL + s);
        if (lane == 0) mbar_arrive_expect_tx(fb, stage_tx);
        __syncwarp();
        const int tok = w.t0 + step * BKT;
        if (lane < 2) tma_load_2d(st + lane * BOX_BYTES, &tm_dy, w.ib * 128 + 64 * lane, tok, fb);
        else if (lane < nbox)
          tma_load_2d(st + STAGE_DY + (lane - 2) * BOX_BYTES, &tm_x, w.jt * BN + 64 * (lane - 2), tok, fb);
        last_g = g;
      }
    }
    // Let every issued copy land before the CTA can exit (the slots this loader used).
    if (lane == 0 && last_g != 0xffffffffu) {
      for (uint32_t k = 0; k < NS && k <= last_g; ++k) {
        const uint32_t gg = last_g - k;
        if (gg % NUM_LOADERS == t) drain_wait(bar(BAR_FULL + gg % NS), (gg / NS) & 1u, args.timeout_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc_g = make_idesc_bf16(128, BN, 1, 1);
      const uint32_t idesc_l = make_idesc_bf16(128, 128, 1, 1);
      const uint32_t idesc_da = make_idesc_bf16(128, args.r16, 0, 0);
      const uint32_t idesc_db = make_idesc_bf16(128, args.r16, 1, 0);
      const int lsteps = args.r16 / 16;
      // Keep this thread's work between MMAs short: stage-0 descriptors are built once;
      // a stage adds STAGE_BYTES / 16 and a 16-token K step adds 2048 bytes (128 units).
      const uint64_t d_dy0 = make_sdesc(smem + OFF_STAGES, BOX_BYTES, 1024, SWZ_128B);
      const uint64_t d_x0 = make_sdesc(smem + OFF_STAGES + STAGE_DY, BOX_BYTES, 1024, SWZ_128B);
      const uint32_t b_full = bar(BAR_FULL), b_empty = bar(BAR_EMPTY);
      uint32_t g = 0, it = 0, cc = 0;
      uint32_t rr = 0;          // NL: rank rounds issued
      uint32_t s = 0, ph = 0;   // stage and phase of global step g
      bool ok = true;
      WorkIter wi = work_begin(args);
      Unit w;
      while (ok && work_next(wi, args, w)) {
        if (!(ok = wait_spin_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 4))) break;
        tc_fence_after();
        for (int step = 0; step < w.nsteps; ++step) {
          if (!(ok = wait_spin_bounded(b_full + 8u * s, ph, ctl, 5))) break;
          tc_fence_after();
          const uint64_t a = d_dy0 + s * (STAGE_BYTES >> 4), b = d_x0 + s * (STAGE_BYTES >> 4);
          static_assert(BKT == 32, "two 16-token K steps per stage");
          mma_bf16(tmem + COL_G, a, b, idesc_g, step > 0 ? 1u : 0u);
          mma_bf16(tmem + COL_G, a + 128, b + 128, idesc_g, 1u);
          mma_commit(b_empty + 8u * s);
          ++g;
          if (++s == NS) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(bar(BAR_ACCFULL));
        if (NL) {
          // dU of the unit written: the code chunk has been read, then the rank rounds
          if (!(ok = wait_spin_bounded(bar(BAR_DUFULL), cc & 1u, ctl, 8))) break;
          tc_fence_after();
          mma_commit(bar(BAR_ECEMPTY));
          const uint32_t idesc_da64 = make_idesc_bf16(128, 64, 0, 0);
          const uint32_t idesc_db64 = make_idesc_bf16(128, 64, 1, 0);
          for (int rc = 0; rc < (args.r16 + 63) / 64; ++rc) {
            // rounds are the uses of the epilogue buffers (EF) in NL
            if (!(ok = wait_spin_bounded(bar(BAR_EFFULL), rr & 1u, ctl, 6))) break;
            const uint32_t b = rr & 1u, n = rr >> 1;
            if (!(ok = wait_spin_bounded(bar(BAR_DRAINED + b), (n & 1u) ^ 1u, ctl, 13))) break;
            tc_fence_after();
            const uint32_t col = tmem + COL_NL + 128u * b;
            // dA round = dU * B_round^T : M = 128 rows i, N = 64 ranks, K = 128 columns j
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              const uint64_t ad = make_sdesc(smem + OFF_DU + 16384u * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
              const uint64_t bd = make_sdesc(smem + OFF_BP + NL_BOX * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
              mma_bf16(col, ad, bd, idesc_da64, ks > 0 ? 1u : 0u);
            }
            // dB^T round = dU^T * A_round : M = 128 columns j (dU MN-major), N = 64 ranks, K = 128 rows i
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              const uint64_t ad = make_sdesc(smem + OFF_DU + 2048u * ks, 16384, 1024, SWZ_128B);
              const uint64_t bd = make_sdesc(smem + OFF_AT + NL_BOX * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
              mma_bf16(col + 64, ad, bd, idesc_db64, ks > 0 ? 1u : 0u);
            }
            mma_commit(bar(b ? BAR_DBFULL1 : BAR_DBFULL));
            mma_commit(bar(BAR_EFEMPTY));
            ++rr;
          }
          if (!ok) break;
          ++cc;
          ++it;
          continue;
        }
        if (!(ok = wait_spin_bounded(bar(BAR_EFFULL), it & 1u, ctl, 6))) break;
        for (int c = 0; c < args.nchunks; ++c) {
          if (!(ok = wait_spin_bounded(bar(BAR_ECFULL), cc & 1u, ctl, 7))) break;
          tc_fence_after();
          // L = A (rows i) * B (columns j of the chunk): both operands read MN-major from
          // A^T and B, 16 rank rows (two 8-row groups) per K step.
          for (int ks = 0; ks < lsteps; ++ks) {
            const uint64_t ad = make_sdesc(smem + OFF_AT + 2048u * ks, rbox, 1024, SWZ_128B);
            const uint64_t bd = make_sdesc(smem + OFF_BP + 2048u * ks, rbox, 1024, SWZ_128B);
            mma_bf16(tmem + COL_L, ad, bd, idesc_l, ks > 0 ? 1u : 0u);
          }
          mma_commit(bar(BAR_LFULL));
          if (!(ok = wait_spin_bounded(bar(BAR_DUFULL), cc & 1u, ctl, 8))) break;
          tc_fence_after();
          // dA (+)= dU * B_chunk^T : M = 128 rows i, N = r16, K = 128 columns j
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t ad = make_sdesc(smem + OFF_DU + 16384u * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
            const uint64_t bd = make_sdesc(smem + OFF_BP + rbox * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
            mma_bf16(tmem + COL_DA, ad, bd, idesc_da, (c > 0 || ks > 0) ? 1u : 0u);
          }
          // dB^T = dU^T * A : M = 128 columns j (dU read MN-major), N = r16, K = 128 rows i
#pragma unroll
          for (int ks = 0; ks < 8; ++ks) {
            const uint64_t ad = make_sdesc(smem + OFF_DU + 2048u * ks, 16384, 1024, SWZ_128B);
            const uint64_t bd = make_sdesc(smem + OFF_AT + rbox * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
            mma_bf16(tmem + COL_DBT, ad, bd, idesc_db, ks > 0 ? 1u : 0u);
          }
          mma_commit(bar(BAR_DBFULL));
          mma_commit(bar(BAR_ECEMPTY));
          ++cc;
        }
        if (!ok) break;
        mma_commit(bar(BAR_EFEMPTY));
        ++it;
      }
      mma_commit(bar(BAR_DRAIN));
      drain_wait(bar(BAR_DRAIN), 0, args.timeout_ns);
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
    uint32_t it = 0, cc = 0;
    uint32_t rr = 0;   // NL: rank rounds drained
    bool ok = true;
    WorkIter wi = work_begin(args);
    Unit w;
    while (ok && work_next(wi, args, w)) {
      const int i_g = w.ib * 128 + row;
      ok = wait_bounded(bar(BAR_ACCFULL), it & 1u, ctl, 9);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      for (int c = 0; c < args.nchunks; ++c) {
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
        // zero offset of the row (group) when the weights are asymmetric (ZP: args.zero set)
        const float z_i = !ZP         ? 0.0f
                          : args.s_ld ? args.zero[static_cast<int64_t>(i_g) * args.s_ld + j0 / args.group_size]
                                      : args.zero[i_g];
        ok = wait_bounded(bar(BAR_ECFULL), cc & 1u, ctl, 10);
        if (!NL) ok = ok && wait_bounded(bar(BAR_LFULL), cc & 1u, ctl, 11);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
        // Packed fp32x2 arithmetic per pair of columns: u = phi^-1 + (alpha/r) L, the
        // unclipped code cu (round half to even by the magic add), the clipped code c,
        // the STE mask M = [c == cu], dU = G * (s_x s) * M and the ds partial sum G * (c - z)
        // (times s_x at the end; z = 0 for symmetric weights).
        const float gs_i = gscale * s_i;
        const float code_n = __fmaf_rn(qp.lo, qp.inv2f, -qp.magic_c);   // n and p as exact floats
        const float code_p = __fmaf_rn(qp.hi, qp.inv2f, -qp.magic_c);
        float2 ds2 = make_float2(0.0f, 0.0f);
#pragma unroll 1
        for (int p = 0; p < 2; ++p) {
          const int jl = 64 * h + 32 * p;   // column within the chunk
          float G[32], Lv[32], v[32];
          tmem_ld32(tmem + lane_off + COL_G + 128 * c + jl, G);
          if (!NL) tmem_ld32(tmem + lane_off + COL_L + jl, Lv);
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
            const float2 u2 = NL   ? v2
                              : UB ? u_bf16x2(Lv[2 * e], Lv[2 * e + 1], v2.x, v2.y, lr2)
                                   : __ffma2_rn(make_float2(Lv[2 * e], Lv[2 * e + 1]),
                                                make_float2(qp.lr_scale, qp.lr_scale), v2);
            const float2 t2 = __fadd2_rn(u2, make_float2(qp.magic, qp.magic));
            const float2 cu = __ffma2_rn(t2, make_float2(qp.inv2f, qp.inv2f), make_float2(-qp.magic_c, -qp.magic_c));
            const float2 cc = make_float2(fminf(fmaxf(cu.x, code_n), code_p), fminf(fmaxf(cu.y, code_n), code_p));
            ds2 = __ffma2_rn(g2, ZP ? __fadd2_rn(cc, make_float2(-z_i, -z_i)) : cc, ds2);
            const float2 gs = __fmul2_rn(g2, make_float2(gs_i, gs_i));
            du[e] = pack_rn_bf16x2(cc.x == cu.x ? gs.x : 0.0f, cc.y == cu.y ? gs.y : 0.0f);
          }
          const uint32_t dub = smem + OFF_DU + 16384u * h;
#pragma unroll
          for (int wq = 0; wq < 4; ++wq)
            st_shared_v4(dub + swz_offset(row, 4 * p + wq, 128), du[4 * wq], du[4 * wq + 1], du[4 * wq + 2],
                         du[4 * wq + 3]);
        }
        if (c == args.nchunks - 1) {
          // Last read of G for this unit: hand the accumulator to the next unit's main
          // loop, which then overlaps the adapter contractions and partial stores below.
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(BAR_ACCEMPTY));
        }
        const float ds_acc = (ds2.x + ds2.y) * gscale;
        // ds partial of this 128-column block (two halves h per row)
        args.ds_part[(static_cast<int64_t>(w.sp * 2 + h) * args.m + i_g) * nb + j0 / 128] = ds_acc;
        tc_fence_before();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_DUFULL));
        if (NL) {
          // rank rounds: this warp half writes 32 of each round's 64 rank columns of dB^T
          // (lanes = columns j) and of dA (lanes = rows i)
          float* dstB = args.dB_part + static_cast<int64_t>(w.ib * args.nsplit + w.sp) * args.r * args.k + j0 + row;
          float* dstA = args.dA_part + (static_cast<int64_t>(w.jt * args.nsplit + w.sp) * args.m + i_g) * args.r;
          for (int rc = 0; rc < (args.r16 + 63) / 64 && ok; ++rc) {
            const uint32_t b = rr & 1u, n = rr >> 1;
            ok = wait_bounded(bar(b ? BAR_DBFULL1 : BAR_DBFULL), n & 1u, ctl, 12);
            if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
            tc_fence_after();
            const uint32_t col = tmem + lane_off + COL_NL + 128u * b + 32u * h;
#pragma unroll 1
            for (int c8 = 0; c8 < 32; c8 += 8) {
              float vb[8], va[8];
              tmem_ld8(col + 64 + c8, vb);
              tmem_ld8(col + c8, va);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 8; ++e) {
                const int t = 64 * rc + 32 * h + c8 + e;
                if (t < args.r) {
                  dstB[static_cast<int64_t>(t) * args.k] = vb[e];
                  dstA[t] = va[e];
                }
              }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(BAR_DRAINED + b));
            ++rr;
          }
          if (!ok) break;
          ++cc;
          continue;
        }
        ok = wait_bounded(bar(BAR_DBFULL), cc & 1u, ctl, 12);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
        // dB^T chunk: lanes = columns j of the chunk, TMEM columns = rank index
        {
          float* dst = args.dB_part + static_cast<int64_t>(w.ib * args.nsplit + w.sp) * args.r * args.k + j0 + row;
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
        if (c == args.nchunks - 1) {
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
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int FMT, bool ZP, bool UB, bool NL = false>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                       const CUtensorMap& e, const DwArgs& args, int grid, cudaStream_t stream) {
  static bool configured[kMaxDevices] = {};
  const cudaError_t err = ensure_smem_attr(reinterpret_cast<const void*>(dw_kernel<FMT, ZP, UB, NL>),
                                           static_cast<int>(SMEM_BYTES), configured);
  if (err != cudaSuccess) return err;
  dw_kernel<FMT, ZP, UB, NL><<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(a, b, c, d, e, args);
  return cudaGetLastError();
}

template <int FMT>
cudaError_t launch_fmt(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                       const CUtensorMap& e, const DwArgs& args, int grid, cudaStream_t stream) {
  if (args.u_bf16) {   // bf16 pre-round value: no zero offsets, bases exact in bf16
    if (FMT == FMT_F16 || args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_one<FMT == FMT_F16 ? FMT_Q8 : FMT, false, true>(a, b, c, d, e, args, grid, stream);
  }
  if (fmt_float(FMT)) {   // zero offsets exist only with the integer formats
    if (args.zero != nullptr) return cudaErrorInvalidValue;
    return launch_one<FMT, false, false>(a, b, c, d, e, args, grid, stream);
  }
  return args.zero != nullptr ? launch_one<FMT, true, false>(a, b, c, d, e, args, grid, stream)
                              : launch_one<FMT, false, false>(a, b, c, d, e, args, grid, stream);
}

}  // namespace

int dw_smem_bytes(int, int) { return static_cast<int>(SMEM_BYTES); }

cudaError_t launch_dw(int fmt, const CUtensorMap& tm_dy, const CUtensorMap& tm_x, const CUtensorMap& tm_at,
                      const CUtensorMap& tm_phi, const CUtensorMap& tm_b, const DwArgs& args, int grid,
                      cudaStream_t stream) {
  if (args.codes_base) {
    // ranks above 64: the base holds int8 codes, 128-column tiles, rank rounds of 64
    if (grid < 1 || fmt != FMT_Q8 || args.u_bf16 || args.nchunks != 1 || args.r16 < 16 || args.r16 > 256 ||
        (args.r16 & 15))
      return cudaErrorInvalidValue;
    return args.zero != nullptr ? launch_one<FMT_Q8, true, false, true>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream)
                                : launch_one<FMT_Q8, false, false, true>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
  }
  if (grid < 1 || args.r16 < 16 || args.r16 > 64 || (args.r16 & 15) || args.nchunks < 1 || args.nchunks > 2)
    return cudaErrorInvalidValue;
  if (fmt_16bit(fmt) && (args.phi == nullptr || (reinterpret_cast<uintptr_t>(args.phi) & 15u) || args.k % 128))
    return cudaErrorInvalidValue;
  switch (fmt) {
    case FMT_Q8: return launch_fmt<FMT_Q8>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    case FMT_I4: return launch_fmt<FMT_I4>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    case FMT_BF16: return launch_fmt<FMT_BF16>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    case FMT_F16: return launch_fmt<FMT_F16>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    case FMT_E4M3: return launch_fmt<FMT_E4M3>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    case FMT_E5M2: return launch_fmt<FMT_E5M2>(tm_dy, tm_x, tm_at, tm_phi, tm_b, args, grid, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace lrqat
