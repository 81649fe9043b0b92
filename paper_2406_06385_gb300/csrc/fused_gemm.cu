// Fused LR-QAT GEMM for the forward (Y = X W_hat^T) and the input gradient
// (dX = dY W_hat), with W_hat rebuilt on chip and never stored (Eq. 8 of the
// paper; the recompute replaces the checkpointing of Sec. 3).
//
// One persistent CTA per SM processes tiles of 128 weight rows x 448 tokens.
// Per 32-wide slice of the contraction:
//   * TMA brings the token operand (448 x 32 bf16, SW64), the stored base
//     (128 x 32 int8, SW32; packed: 128 x 16 bytes) and a 32-row slice of the
//     second low-rank factor (SW128).
//   * The MMA warp computes the low-rank tile L = RF * SF^T (M=128, N=32,
//     K=r rounded to 16) into TMEM with tcgen05.
//   * Eight producer warps read L from TMEM, decode the stored base, form
//     u = phi^{-1}(Phi0) + (alpha/r) L, round half to even, clip, (scale) and
//     write the bf16 operand tile (SW64, K-major) into shared memory.
//   * The MMA warp runs the main product into two 128 x 224 fp32 TMEM
//     accumulators; the same eight warps drain them in the epilogue.
// Forward: rows = m (weight rows), contraction = k, RF = A (padded), SF = B^T.
// dX:      rows = k, contraction = m over the transposed base Phi0^T,
//          RF = B^T (padded), SF = A (padded); the scale varies along the
//          contraction, so the producer emits bf16(s * c).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int BM = 128;
constexpr int BK = 32;
constexpr int BN = 224;
constexpr int NACC = 2;
constexpr int BT = BN * NACC;
constexpr int NS = 4;
constexpr int NUM_THREADS = 320;
constexpr int NUM_PROD_WARPS = 8;

constexpr uint32_t RF_BYTES = 128 * 128;
constexpr uint32_t TOK_HALF = BN * 64;
constexpr uint32_t TOK_BYTES = BT * 64;
constexpr uint32_t W_BYTES = 128 * 64;
constexpr uint32_t PHI_BYTES = 128 * 32;
constexpr uint32_t SF_BYTES = 32 * 128;
constexpr uint32_t OFF_TOK = 0;
constexpr uint32_t OFF_W = TOK_BYTES;
constexpr uint32_t OFF_PHI = OFF_W + W_BYTES;
constexpr uint32_t OFF_SF = OFF_PHI + PHI_BYTES;
constexpr uint32_t STAGE_BYTES = OFF_SF + SF_BYTES;
constexpr uint32_t OFF_RF = 0;
constexpr uint32_t OFF_STAGES = RF_BYTES;
constexpr uint32_t SMEM_BYTES = OFF_STAGES + NS * STAGE_BYTES + 1024;   // + 1 KB for 1024-B alignment

static_assert(STAGE_BYTES % 1024 == 0 && TOK_HALF % 1024 == 0 && OFF_W % 1024 == 0 && OFF_PHI % 1024 == 0 &&
                  OFF_SF % 1024 == 0,
              "swizzled tiles must start on 1024-byte boundaries");

constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t COL_L = NACC * BN;   // two 32-column low-rank buffers at 448 and 480
static_assert(COL_L + 2 * BK <= TMEM_COLS, "TMEM budget");

// barrier indices
constexpr int BAR_FULL = 0;
constexpr int BAR_EMPTY = BAR_FULL + NS;
constexpr int BAR_WFULL = BAR_EMPTY + NS;
constexpr int BAR_LFULL = BAR_WFULL + NS;
constexpr int BAR_LEMPTY = BAR_LFULL + 2;
constexpr int BAR_RFFULL = BAR_LEMPTY + 2;
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

template <int MODE, bool PACKED>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    fused_gemm_kernel(const __grid_constant__ CUtensorMap tm_tok, const __grid_constant__ CUtensorMap tm_phi,
                      const __grid_constant__ CUtensorMap tm_rf, const __grid_constant__ CUtensorMap tm_sf,
                      const FusedArgs args) {
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
    for (int s = 0; s < NS; ++s) {
      mbar_init(bar(BAR_FULL + s), 1);
      mbar_init(bar(BAR_EMPTY + s), 1);
      mbar_init(bar(BAR_WFULL + s), NUM_PROD_WARPS);
    }
    for (int b = 0; b < 2; ++b) {
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
  if (warp == 1) tmem_alloc(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};
  const int nk = args.kdim / BK;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tm_tok);
      prefetch_tensormap(&tm_phi);
      prefetch_tensormap(&tm_rf);
      prefetch_tensormap(&tm_sf);
      const uint32_t stage_tx = TOK_BYTES + (PACKED ? PHI_BYTES / 2 : PHI_BYTES) + SF_BYTES;
      uint32_t g = 0;
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
        const int rb = tile % args.num_rb;
        const int tb = tile / args.num_rb;
        if (!(ok = wait_bounded(bar(BAR_RFEMPTY), (it & 1u) ^ 1u, ctl, 1))) break;
        mbar_arrive_expect_tx(bar(BAR_RFFULL), RF_BYTES);
        tma_load_2d(smem + OFF_RF, &tm_rf, 0, rb * BM, bar(BAR_RFFULL));
        ++it;
        for (int kk = 0; kk < nk; ++kk) {
          const uint32_t s = g % NS, ph = (g / NS) & 1u;
          if (!(ok = wait_bounded(bar(BAR_EMPTY + s), ph ^ 1u, ctl, 2))) break;
          const uint32_t st = smem + OFF_STAGES + s * STAGE_BYTES;
          const uint32_t fb = bar(BAR_FULL + s);
          mbar_arrive_expect_tx(fb, stage_tx);
          tma_load_2d(st + OFF_TOK, &tm_tok, kk * BK, tb * BT, fb);
          tma_load_2d(st + OFF_TOK + TOK_HALF, &tm_tok, kk * BK, tb * BT + BN, fb);
          tma_load_2d(st + OFF_PHI, &tm_phi, PACKED ? kk * (BK / 2) : kk * BK, rb * BM, fb);
          tma_load_2d(st + OFF_SF, &tm_sf, 0, kk * BK, fb);
          ++g;
        }
      }
      // Let every issued copy land before the CTA can exit.
      for (uint32_t s = 0; s < NS && s < g; ++s) {
        const uint32_t last = s + NS * ((g - 1 - s) / NS);
        drain_wait(bar(BAR_FULL + s), (last / NS) & 1u, args.timeout_ns);
      }
      if (it > 0) drain_wait(bar(BAR_RFFULL), (it - 1) & 1u, args.timeout_ns);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc_main = make_idesc_bf16(128, BN, 0, 0);
      const uint32_t idesc_l = make_idesc_bf16(128, BK, 0, 0);
      const int lsteps = args.r16 / 16;
      uint32_t g = 0;
      uint32_t it = 0;
      bool ok = true;
      auto issue_lowrank = [&](uint32_t gg) -> bool {
        const uint32_t s = gg % NS, ph = (gg / NS) & 1u;
        const uint32_t lb = gg & 1u, lph = (gg >> 1) & 1u;
        if (!wait_bounded(bar(BAR_FULL + s), ph, ctl, 3)) return false;
        if (!wait_bounded(bar(BAR_LEMPTY + lb), lph ^ 1u, ctl, 4)) return false;
        tc_fence_after();
        const uint32_t sf = smem + OFF_STAGES + s * STAGE_BYTES + OFF_SF;
        for (int ks = 0; ks < lsteps; ++ks) {
          const uint64_t ad = make_sdesc(smem + OFF_RF + 32u * ks, 16, 1024, SWZ_128B);
          const uint64_t bd = make_sdesc(sf + 32u * ks, 16, 1024, SWZ_128B);
          mma_bf16(tmem + COL_L + BK * lb, ad, bd, idesc_l, ks > 0 ? 1u : 0u);
        }
        mma_commit(bar(BAR_LFULL + lb));
        return true;
      };
      for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
        if (!(ok = wait_bounded(bar(BAR_RFFULL), it & 1u, ctl, 5))) break;
        if (!(ok = issue_lowrank(g))) break;
        if (nk == 1) mma_commit(bar(BAR_RFEMPTY));
        if (!(ok = wait_bounded(bar(BAR_ACCEMPTY), (it & 1u) ^ 1u, ctl, 6))) break;
        tc_fence_after();
        for (int kk = 0; kk < nk; ++kk) {
          const uint32_t gg = g + kk;
          if (kk + 1 < nk) {
            if (!(ok = issue_lowrank(gg + 1))) break;
            if (kk + 2 == nk) mma_commit(bar(BAR_RFEMPTY));
          }
          const uint32_t s = gg % NS, ph = (gg / NS) & 1u;
          if (!(ok = wait_bounded(bar(BAR_WFULL + s), ph, ctl, 7))) break;
          tc_fence_after();
          const uint32_t st = smem + OFF_STAGES + s * STAGE_BYTES;
#pragma unroll
          for (int a = 0; a < NACC; ++a) {
#pragma unroll
            for (int ks = 0; ks < BK / 16; ++ks) {
              const uint64_t ad = make_sdesc(st + OFF_W + 32u * ks, 16, 512, SWZ_64B);
              const uint64_t bd = make_sdesc(st + OFF_TOK + a * TOK_HALF + 32u * ks, 16, 512, SWZ_64B);
              mma_bf16(tmem + a * BN, ad, bd, idesc_main, (kk > 0 || ks > 0) ? 1u : 0u);
            }
          }
          mma_commit(bar(BAR_EMPTY + s));
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
    const int pw = warp - 2;
    const int q = warp & 3;           // TMEM lane quarter this warp may access
    const int h = pw >> 2;            // half of the slice columns / accumulator index
    const int row = q * 32 + lane;    // row of the tile handled by this thread
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const QuantParams qp = args.q;
    uint32_t g = 0;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < args.num_tiles && ok; tile += gridDim.x) {
      const int rb = tile % args.num_rb;
      const int tb = tile / args.num_rb;
      const int row_g = rb * BM + row;
      for (int kk = 0; kk < nk; ++kk) {
        const uint32_t gg = g + kk;
        const uint32_t s = gg % NS, ph = (gg / NS) & 1u;
        const uint32_t lb = gg & 1u, lph = (gg >> 1) & 1u;
        // Scales that multiply the operand (group-wise forward, dX).
        float sc[16];
        if (MODE == FUSED_FWD_GROUP) {
          const float v = args.s[static_cast<int64_t>(row_g) * args.s_ld + (kk * BK) / args.group_size];
#pragma unroll
          for (int e = 0; e < 16; ++e) sc[e] = v;
        } else if (MODE == FUSED_DX) {
          const int i0 = kk * BK + 16 * h;
          if (args.s_ld == 0) {
            const float4* sp = reinterpret_cast<const float4*>(args.s + i0);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float4 v = __ldg(sp + e);
              sc[4 * e] = v.x;
              sc[4 * e + 1] = v.y;
              sc[4 * e + 2] = v.z;
              sc[4 * e + 3] = v.w;
            }
          } else {
            const int gcol = row_g / args.group_size;
#pragma unroll
            for (int e = 0; e < 16; ++e) sc[e] = __ldg(args.s + static_cast<int64_t>(i0 + e) * args.s_ld + gcol);
          }
        }
        ok = wait_bounded(bar(BAR_LFULL + lb), lph, ctl, 8);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        tc_fence_after();
        float Lv[16];
        tmem_ld16(tmem + lane_off + COL_L + BK * lb + 16 * h, Lv);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_LEMPTY + lb));
        ok = wait_bounded(bar(BAR_FULL + s), ph, ctl, 9);
        if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
        const uint32_t st = smem + OFF_STAGES + s * STAGE_BYTES;
        float v[16];
        if (PACKED) {
          const uint2 raw = ld_shared_v2(st + OFF_PHI + row * 16 + 8 * h);
          decode_i4x8(raw.x, v);
          decode_i4x8(raw.y, v + 8);
        } else {
          const uint4 raw = ld_shared_v4(st + OFF_PHI + swz_offset(row, h, 32));
          decode_i8x4(raw.x, v);
          decode_i8x4(raw.y, v + 4);
          decode_i8x4(raw.z, v + 8);
          decode_i8x4(raw.w, v + 12);
        }
        uint32_t w[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float c0 = lrqat_code(Lv[2 * e], v[2 * e], qp);
          const float c1 = lrqat_code(Lv[2 * e + 1], v[2 * e + 1], qp);
          if (MODE == FUSED_FWD_PC)
            w[e] = pack_exact_bf16x2(c0, c1);
          else
            w[e] = pack_rn_bf16x2(c0 * sc[2 * e], c1 * sc[2 * e + 1]);
        }
        const uint32_t wt = st + OFF_W;
        st_shared_v4(wt + swz_offset(row, 2 * h, 64), w[0], w[1], w[2], w[3]);
        st_shared_v4(wt + swz_offset(row, 2 * h + 1, 64), w[4], w[5], w[6], w[7]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_WFULL + s));
      }
      if (!ok) break;
      // ------------------------------------------------------------ epilogue
      float scale = 1.0f;
      if (MODE == FUSED_FWD_PC) scale = args.s[row_g];
      if (MODE != FUSED_DX && args.s_x != nullptr) scale *= *args.s_x;
      ok = wait_bounded(bar(BAR_ACCFULL), it & 1u, ctl, 10);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float acc[32];
        tmem_ld32(tmem + lane_off + h * BN + 32 * c, acc);
        tmem_ld_wait();
        const int tok0 = tb * BT + h * BN + 32 * c;
        uint32_t mword = 0xffffffffu;
        if (MODE == FUSED_DX && args.xmask != nullptr && tok0 < args.T)
          mword = args.xmask[static_cast<int64_t>(row_g) * args.xmask_ld + tok0 / 32];
        uint16_t* dst = args.out + static_cast<int64_t>(tok0) * args.out_ld + row_g;
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          if (tok0 + e < args.T) {
            const float val = ((mword >> e) & 1u) ? acc[e] * scale : 0.0f;
            dst[static_cast<int64_t>(e) * args.out_ld] = float_to_bf16_rn(val);
          }
        }
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

template <int MODE, bool PACKED>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& d,
                       const FusedArgs& args, int grid, cudaStream_t stream) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(fused_gemm_kernel<MODE, PACKED>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  fused_gemm_kernel<MODE, PACKED><<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(a, b, c, d, args);
  return cudaGetLastError();
}

}  // namespace

int fused_smem_bytes() { return static_cast<int>(SMEM_BYTES); }

cudaError_t launch_fused(int mode, int packed, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi,
                         const CUtensorMap& tm_rf, const CUtensorMap& tm_sf, const FusedArgs& args, int grid,
                         cudaStream_t stream) {
  if (grid < 1) return cudaErrorInvalidValue;
  switch (mode) {
    case FUSED_FWD_PC:
      return packed ? launch_one<FUSED_FWD_PC, true>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream)
                    : launch_one<FUSED_FWD_PC, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FUSED_FWD_GROUP:
      return packed ? launch_one<FUSED_FWD_GROUP, true>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream)
                    : launch_one<FUSED_FWD_GROUP, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    case FUSED_DX:
      return launch_one<FUSED_DX, false>(tm_tok, tm_phi, tm_rf, tm_sf, args, grid, stream);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace lrqat
