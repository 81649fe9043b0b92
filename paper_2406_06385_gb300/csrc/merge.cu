// Merge on the tensor cores (Sec. 3: after training the integer weight is
// W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p), and W_hat = s W_Z), and the
// same pass writing the unclipped codes for the GEMMs of ranks above 64.
//
// One CTA of four warps per 128 x 128 tile: the tile's rows of A and columns of B land
// by TMA, r16 / 16 tcgen05 MMAs write the low-rank tile L = A B into TMEM, and warp q
// turns rows 32q .. 32q + 31 into codes (TMEM lane = row): it reads L 32 columns at a
// time, decodes the stored base of the same 32 columns from global memory, rounds,
// clamps to [lo, hi] of the quantizer constants and stores 32 int8 codes as two 16-byte
// words.  The pass moves the base and the codes once (the product costs 2 m k r flops
// on the tensor cores instead of the CUDA cores).
//   A operand: K-major boxes of 64 rank columns read from A [m, r] (r % 8 == 0; columns
//   past r read as zeros), or (AMN) two MN-major boxes of r16 rank rows x 64 rows read
//   from the zero-padded A^T [r16, m].
//   B operand: two MN-major boxes of r16 rank rows x 64 columns read from B [r, k] (rows
//   past r read as zeros) or from the zero-padded B [r16, k].
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "merge.h"
#include "ptx.cuh"
#include "quant.cuh"

namespace lrqat {
namespace {

// A: up to 64 KB (r16 = 256), then B: two boxes of r16 rows x 128 bytes.  Small ranks
// pad the allocation to 52 KB so that at most four CTAs share an SM: four 128-column
// TMEM allocations fill its 512 columns, and a fifth CTA would wait inside
// tcgen05.alloc (ranks above 64 need more shared memory, so fewer CTAs fit anyway).
constexpr uint32_t MIN_SMEM_BYTES = 52 * 1024;
constexpr uint32_t MAX_SMEM_BYTES = 2 * 65536 + 1024;
constexpr uint32_t TMEM_COLS = 128;

__host__ __device__ constexpr uint32_t a_tile_bytes(int r16, bool amn) {
  return amn ? 2u * 128u * static_cast<uint32_t>(r16) : 16384u * static_cast<uint32_t>((r16 + 63) / 64);
}
__host__ __device__ constexpr uint32_t smem_bytes(int r16, bool amn) {
  return a_tile_bytes(r16, amn) + 2u * 128u * static_cast<uint32_t>(r16) + 1024u < MIN_SMEM_BYTES
             ? MIN_SMEM_BYTES
             : a_tile_bytes(r16, amn) + 2u * 128u * static_cast<uint32_t>(r16) + 1024u;
}

// Raw words of the stored base per 32 columns of a row: 16 bytes (packed nibbles),
// 32 bytes (one byte per value) or 64 bytes (16-bit values).
template <int FMT>
__host__ __device__ constexpr int raw_words() { return FMT == FMT_I4 ? 4 : fmt_16bit(FMT) ? 16 : 8; }
// Chunks of 32 columns whose raw words are in flight at once: all four of the tile,
// or two for the 16-bit bases (whose words would otherwise cost 64 registers).
template <int FMT>
__host__ __device__ constexpr int prefetch_depth() { return fmt_16bit(FMT) ? 2 : 4; }

// Raw words of columns col0 .. col0 + 31 of row `row` (16-byte loads).
template <int FMT>
__device__ __forceinline__ void load_raw32(const void* phi0, int64_t row, int64_t k, int64_t col0, uint32_t* w) {
  constexpr int NV = raw_words<FMT>() / 4;
  const uint8_t* base = static_cast<const uint8_t*>(phi0);
  const int64_t off = FMT == FMT_I4 ? row * (k / 2) + col0 / 2 : fmt_16bit(FMT) ? 2 * (row * k + col0) : row * k + col0;
  const uint4* src = reinterpret_cast<const uint4*>(base + off);
#pragma unroll
  for (int e = 0; e < NV; ++e) {
    const uint4 a = __ldg(src + e);
    w[4 * e] = a.x, w[4 * e + 1] = a.y, w[4 * e + 2] = a.z, w[4 * e + 3] = a.w;
  }
}

// The raw words of 32 columns -> v[32] in the units of u_f.
template <int FMT>
__device__ __forceinline__ void decode32(const uint32_t* w, float (&v)[32]) {
  decode16<FMT>(w, v);
  decode16<FMT>(w + raw_words<FMT>() / 2, v + 16);
}

template <int FMT, bool UB, bool AMN>
__global__ void __launch_bounds__(128) merge_tc_kernel(const __grid_constant__ CUtensorMap tm_a,
                                                       const __grid_constant__ CUtensorMap tm_b, const MergeArgs args) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[2];   // operands landed, low-rank tile done
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int abort_s;
  const uint32_t smem = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t rb = blockIdx.y, cb = blockIdx.x;
  const uint32_t bar_load = smem_u32(&bars[0]), bar_mma = smem_u32(&bars[1]);
  // This thread's row of the tile: its stored base is requested first, so that the loads
  // overlap the operand copies and the MMAs.
  const int64_t row = rb * 128 + 32 * warp + lane;
  constexpr int NW = raw_words<FMT>(), PD = prefetch_depth<FMT>();
  uint32_t raw[PD][NW];
#pragma unroll
  for (int cc = 0; cc < PD; ++cc) load_raw32<FMT>(args.phi0, row, args.k, cb * 128 + 32 * cc, raw[cc]);
  if (threadIdx.x == 0) {
    abort_s = 0;
    mbar_init(bar_load, 1);
    mbar_init(bar_mma, 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};
  const int r16 = args.r16;
  const uint32_t rbox = 128u * static_cast<uint32_t>(r16);   // bytes of one r16-row x 64-column box
  const uint32_t off_b = a_tile_bytes(r16, AMN);
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(bar_load, off_b + 2u * rbox);
    if (AMN) {
      tma_load_2d(smem, &tm_a, static_cast<int32_t>(rb * 128), 0, bar_load);
      tma_load_2d(smem + rbox, &tm_a, static_cast<int32_t>(rb * 128 + 64), 0, bar_load);
    } else {
      for (int kb = 0; kb < (r16 + 63) / 64; ++kb)
        tma_load_2d(smem + 16384u * kb, &tm_a, 64 * kb, static_cast<int32_t>(rb * 128), bar_load);
    }
    tma_load_2d(smem + off_b, &tm_b, static_cast<int32_t>(cb * 128), 0, bar_load);
    tma_load_2d(smem + off_b + rbox, &tm_b, static_cast<int32_t>(cb * 128 + 64), 0, bar_load);
    if (wait_bounded(bar_load, 0, ctl, 1)) {
      tc_fence_after();
      // A K-major: 32 bytes per 16-element K step inside a 64-column box, one box (16 KB)
      // per 64 ranks; A and B MN-major: two 64-wide atoms (LBO = one box), 16 rank rows =
      // 2048 bytes per K step.
      const uint32_t idesc = make_idesc_bf16(128, 128, AMN ? 1 : 0, 1);
      const uint64_t db = make_sdesc(smem + off_b, rbox, 1024, SWZ_128B);
      for (int ks = 0; ks < r16 / 16; ++ks) {
        const uint64_t da = AMN ? make_sdesc(smem + 2048u * ks, rbox, 1024, SWZ_128B)
                                : make_sdesc(smem + 16384u * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
        mma_bf16(tmem, da, db + 128 * ks, idesc, ks > 0 ? 1u : 0u);
      }
      mma_commit(bar_mma);
    }
  }
  __syncwarp();
  bool ok = wait_bounded(bar_mma, 0, ctl, 2);
  if (__all_sync(0xffffffffu, ok)) {
    tc_fence_after();
    const QuantParams q = args.q;
    const uint32_t lr2 = pack_rn_bf16x2(q.lr_scale, q.lr_scale);   // exact: a power of two when UB
    const uint32_t lane_off = static_cast<uint32_t>(32 * warp) << 16;
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
      const int64_t col0 = cb * 128 + 32 * cc;
      float v[32], L[32];
      decode32<FMT>(raw[cc % PD], v);
      if (cc + PD < 4) load_raw32<FMT>(args.phi0, row, args.k, col0 + 32 * PD, raw[cc % PD]);
      tmem_ld32(tmem + lane_off + 32u * cc, L);
      tmem_ld_wait();
      uint32_t o[8];
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        uint32_t word = 0;
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int i = 4 * g + e;
          float c0, c1;
          if (UB) {
            const float2 u = u_bf16x2(L[i], L[i + 1], v[i], v[i + 1], lr2);
            c0 = code_from_magic(__fadd_rn(u.x, q.magic), q);
            c1 = code_from_magic(__fadd_rn(u.y, q.magic), q);
          } else {
            c0 = lrqat_code(L[i], v[i], q);
            c1 = lrqat_code(L[i + 1], v[i + 1], q);
          }
          word |= (static_cast<uint32_t>(__float2int_rn(c0)) & 0xFFu) << (8 * e);
          word |= (static_cast<uint32_t>(__float2int_rn(c1)) & 0xFFu) << (8 * e + 8);
        }
        o[g] = word;
      }
      uint4* dst = reinterpret_cast<uint4*>(args.wz + row * args.k + col0);
      dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
      dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
    }
  } else if (threadIdx.x == 0) {
    // gave up: let the operand copies land before the CTA (and its shared memory) ends
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(bar_load, 0) && global_timer_ns() - t0 < args.timeout_ns) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int FMT, bool UB, bool AMN>
cudaError_t launch_merge_one(const CUtensorMap& tm_a, const CUtensorMap& tm_b, const MergeArgs& args,
                             cudaStream_t stream) {
  static bool configured[kMaxDevices] = {};
  const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(merge_tc_kernel<FMT, UB, AMN>),
                                         static_cast<int>(MAX_SMEM_BYTES), configured);
  if (e != cudaSuccess) return e;
  dim3 grid(static_cast<unsigned>(args.k / 128), static_cast<unsigned>(args.m / 128));
  merge_tc_kernel<FMT, UB, AMN><<<grid, 128, smem_bytes(args.r16, AMN), stream>>>(tm_a, tm_b, args);
  return cudaGetLastError();
}

template <bool UB, bool AMN>
cudaError_t launch_merge_ub(int fmt, const CUtensorMap& tm_a, const CUtensorMap& tm_b, const MergeArgs& args,
                            cudaStream_t stream) {
  switch (fmt) {
    case FMT_Q8: return launch_merge_one<FMT_Q8, UB, AMN>(tm_a, tm_b, args, stream);
    case FMT_I4: return launch_merge_one<FMT_I4, UB, AMN>(tm_a, tm_b, args, stream);
    case FMT_BF16: return launch_merge_one<FMT_BF16, UB, AMN>(tm_a, tm_b, args, stream);
    case FMT_F16: return UB ? cudaErrorInvalidValue : launch_merge_one<FMT_F16, false, AMN>(tm_a, tm_b, args, stream);
    case FMT_E4M3: return launch_merge_one<FMT_E4M3, UB, AMN>(tm_a, tm_b, args, stream);
    case FMT_E5M2: return launch_merge_one<FMT_E5M2, UB, AMN>(tm_a, tm_b, args, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

static_assert(smem_bytes(256, true) <= MAX_SMEM_BYTES && smem_bytes(256, false) <= MAX_SMEM_BYTES, "smem budget");

cudaError_t launch_merge_tc(int fmt, int u_bf16, int a_mn, const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const MergeArgs& args, cudaStream_t stream) {
  if (args.m % 128 || args.k % 128 || args.r16 < 16 || args.r16 > 256 || (args.r16 & 15)) return cudaErrorInvalidValue;
  if (a_mn) return u_bf16 ? launch_merge_ub<true, true>(fmt, tm_a, tm_b, args, stream)
                          : launch_merge_ub<false, true>(fmt, tm_a, tm_b, args, stream);
  return u_bf16 ? launch_merge_ub<true, false>(fmt, tm_a, tm_b, args, stream)
                : launch_merge_ub<false, false>(fmt, tm_a, tm_b, args, stream);
}

}  // namespace lrqat
