// Merge on the tensor cores (Sec. 3: after training the integer weight is
// W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p), and W_hat = s W_Z), and the
// same pass writing the one-byte codes that the fused GEMMs read as their base (the codes
// path): the clipped code plus a bias (64, or 128 for 8-bit weights) where only the forward
// and dX GEMMs read them, the unclipped code saturated to int8 where dW needs the clip mask
// (ranks above 64).
//
// Tiles of 128 x 128: the tile's rows of A and columns of B land by TMA, r16 / 16 tcgen05
// MMAs write the low-rank tile L = A B into TMEM, and warp q turns rows 32q .. 32q + 31 into
// codes (TMEM lane = row): it reads L 32 columns at a time, takes the stored base of the same
// 32 columns (staged by TMA into the operand slot), rounds, clamps to [lo, hi] of the quantizer
// constants, adds the bias and stores 32 one-byte codes as two 16-byte words.  The CTAs are persistent and overlap one tile's
// codes with the next tile's copies and MMAs (two TMEM buffers).  The pass moves the base and the codes once (the product costs 2 m k r flops
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

// Operand slot: A (up to 64 KB at r16 = 256), then B (two boxes of r16 rows x 128 bytes).
// Two slots when they fit (ranks up to 128), else one.  Every CTA asks for at least 80 KB of
// shared memory so that no more than two CTAs share an SM: two 256-column TMEM allocations
// fill its 512 columns, and a third CTA would wait inside tcgen05.alloc.
constexpr uint32_t MIN_SMEM_BYTES = 80 * 1024;
constexpr uint32_t MAX_SMEM_BYTES = 232448 - 1024;   // the per-CTA limit, less the static barriers
constexpr uint32_t TMEM_COLS = 256;   // two 128-column low-rank tiles
constexpr int NUM_EPI_WARPS = 4;
constexpr int NUM_THREADS = 32 * (NUM_EPI_WARPS + 1);   // + the TMA / MMA warp

__host__ __device__ constexpr uint32_t a_tile_bytes(int r16, bool amn) {
  return amn ? 2u * 128u * static_cast<uint32_t>(r16) : 16384u * static_cast<uint32_t>((r16 + 63) / 64);
}
// Bytes of the stored base of a 128 x 128 tile: 8-bit values, packed nibbles, 16-bit values.
__host__ __device__ constexpr uint32_t phi_tile_bytes(int fmt) {
  return fmt == FMT_I4 ? 8192u : fmt_16bit(fmt) ? 32768u : 16384u;
}
// Operand slot: A, then B, then the stored base of the tile.
__host__ __device__ constexpr uint32_t slot_bytes(int r16, bool amn, int fmt) {
  return a_tile_bytes(r16, amn) + 2u * 128u * static_cast<uint32_t>(r16) + phi_tile_bytes(fmt);
}
// Slots: as many (up to four) as fit while two CTAs share an SM; when not even two fit, as
// many as fit in one CTA per SM.
constexpr uint32_t MAX_SLOTS = 4;
constexpr uint32_t TWO_PER_SM_BYTES = 232448u / 2u - 1024u;
__host__ __device__ constexpr uint32_t min_u(uint32_t a, uint32_t b) { return a < b ? a : b; }
__host__ __device__ constexpr int num_slots(int r16, bool amn, int fmt) {
  return (TWO_PER_SM_BYTES - 1024u) / slot_bytes(r16, amn, fmt) >= 2
             ? static_cast<int>(min_u(MAX_SLOTS, (TWO_PER_SM_BYTES - 1024u) / slot_bytes(r16, amn, fmt)))
             : static_cast<int>(min_u(MAX_SLOTS, (MAX_SMEM_BYTES - 1024u) / slot_bytes(r16, amn, fmt)));
}
__host__ __device__ constexpr uint32_t smem_bytes(int r16, bool amn, int fmt) {
  return num_slots(r16, amn, fmt) * slot_bytes(r16, amn, fmt) + 1024u < MIN_SMEM_BYTES
             ? MIN_SMEM_BYTES
             : num_slots(r16, amn, fmt) * slot_bytes(r16, amn, fmt) + 1024u;
}

__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > timeout_ns) break;
  }
}

// Raw words of the stored base per 32 columns of a row: 16 bytes (packed nibbles),
// 32 bytes (one byte per value) or 64 bytes (16-bit values).
template <int FMT>
__host__ __device__ constexpr int raw_words() { return FMT == FMT_I4 ? 4 : fmt_16bit(FMT) ? 16 : 8; }

// Raw words of columns 32 cc .. 32 cc + 31 of row `row` of the base tile in shared memory, as
// TMA wrote it: 128-byte rows (SW128) of 8-bit values, 64-byte rows (SW64) of nibbles, or two
// 64-column boxes of 128-byte rows (SW128) of 16-bit values.
template <int FMT>
__device__ __forceinline__ void lds_raw32(uint32_t tile, uint32_t row, int cc, uint32_t* w) {
  constexpr int NV = raw_words<FMT>() / 4;
#pragma unroll
  for (int e = 0; e < NV; ++e) {
    uint32_t addr;
    if (FMT == FMT_I4) addr = tile + swz_offset(row, cc, 64);
    else if (fmt_16bit(FMT)) addr = tile + 16384u * (cc >> 1) + swz_offset(row, 4 * (cc & 1) + e, 128);
    else addr = tile + swz_offset(row, 2 * cc + e, 128);
    const uint4 a = ld_shared_v4(addr);
    w[4 * e] = a.x, w[4 * e + 1] = a.y, w[4 * e + 2] = a.z, w[4 * e + 3] = a.w;
  }
}

// The raw words of 32 columns -> v[32] in the units of u_f.
template <int FMT>
__device__ __forceinline__ void decode32(const uint32_t* w, float (&v)[32]) {
  decode16<FMT>(w, v);
  decode16<FMT>(w + raw_words<FMT>() / 2, v + 16);
}

// Persistent: CTA b takes the 128 x 128 tiles b, b + gridDim.x, ... (column tile fastest).
// Warp 4 brings tile i's A rows, B columns and stored base into operand slot i % NSLOT by TMA
// and issues its r16 / 16 MMAs into TMEM buffer i % 2 (128 columns); warps 0-3 turn tile
// i - 1's buffer into codes meanwhile.  Warp q of the epilogue owns rows 32q .. 32q + 31
// (TMEM lane = row).  A slot is refilled once the epilogue has read the tile's base (which is
// after the tile's MMAs completed).
template <int FMT, bool UB, bool AMN>
__global__ void __launch_bounds__(NUM_THREADS) merge_tc_kernel(const __grid_constant__ CUtensorMap tm_a,
                                                               const __grid_constant__ CUtensorMap tm_b,
                                                               const __grid_constant__ CUtensorMap tm_phi,
                                                               const MergeArgs args) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[2 * MAX_SLOTS + 5];   // FULL[4], SEMPTY[4], LFULL[2], LEMPTY[2], DRAIN
  __shared__ uint32_t tmem_base_s;
  __shared__ volatile int abort_s;
  const uint32_t smem = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  auto bar = [&](int i) { return smem_u32(&bars[i]); };
  constexpr int B_FULL = 0, B_SEMPTY = MAX_SLOTS, B_LFULL = 2 * MAX_SLOTS, B_LEMPTY = B_LFULL + 2,
                B_DRAIN = B_LEMPTY + 2;
  const int r16 = args.r16;
  const int nslot = num_slots(r16, AMN, FMT);
  const int64_t nkb = args.k / 128;
  const int64_t num_tiles = (args.m / 128) * nkb;
  if (threadIdx.x == 0) {
    abort_s = 0;
    for (uint32_t i = 0; i < MAX_SLOTS; ++i) {
      mbar_init(bar(B_FULL + i), 1);
      mbar_init(bar(B_SEMPTY + i), NUM_EPI_WARPS);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(B_LFULL + i), 1);
      mbar_init(bar(B_LEMPTY + i), NUM_EPI_WARPS);
    }
    mbar_init(bar(B_DRAIN), 1);
    mbar_fence_init();
  }
  if (warp == NUM_EPI_WARPS) tmem_alloc(smem_u32(&tmem_base_s), TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  const WaitCtl ctl{&abort_s, args.status, args.timeout_ns};

  if (warp == NUM_EPI_WARPS) {
    // ------------------------------------------------------------ TMA + MMA
    if (lane == 0) {
      prefetch_tensormap(&tm_a);
      prefetch_tensormap(&tm_b);
      prefetch_tensormap(&tm_phi);
      const uint32_t rbox = 128u * static_cast<uint32_t>(r16);   // one r16-row x 64-column box
      const uint32_t off_b = a_tile_bytes(r16, AMN), sbytes = slot_bytes(r16, AMN, FMT);
      const uint32_t off_phi = off_b + 2u * rbox;
      // A K-major: 32 bytes per 16-element K step inside a 64-column box, one box (16 KB)
      // per 64 ranks; A and B MN-major: two 64-wide atoms (LBO = one box), 16 rank rows =
      // 2048 bytes per K step.
      const uint32_t idesc = make_idesc_bf16(128, 128, AMN ? 1 : 0, 1);
      bool ok = true, pending = false;   // pending: a copy whose FULL phase was not waited for
      uint32_t i = 0, pend_sl = 0, pend_par = 0;
      for (int64_t t = blockIdx.x; t < num_tiles && ok; t += gridDim.x, ++i) {
        const int64_t rb = t / nkb, cb = t % nkb;
        const uint32_t sl = i % nslot, su = i / nslot, b = i & 1u, bu = i >> 1;
        const uint32_t sa = smem + sl * sbytes;
        if (!(ok = wait_spin_bounded(bar(B_SEMPTY + sl), (su & 1u) ^ 1u, ctl, 1))) break;
        mbar_arrive_expect_tx(bar(B_FULL + sl), sbytes);
        if (AMN) {
          tma_load_2d(sa, &tm_a, static_cast<int32_t>(rb * 128), 0, bar(B_FULL + sl));
          tma_load_2d(sa + rbox, &tm_a, static_cast<int32_t>(rb * 128 + 64), 0, bar(B_FULL + sl));
        } else {
          for (int kb = 0; kb < (r16 + 63) / 64; ++kb)
            tma_load_2d(sa + 16384u * kb, &tm_a, 64 * kb, static_cast<int32_t>(rb * 128), bar(B_FULL + sl));
        }
        tma_load_2d(sa + off_b, &tm_b, static_cast<int32_t>(cb * 128), 0, bar(B_FULL + sl));
        tma_load_2d(sa + off_b + rbox, &tm_b, static_cast<int32_t>(cb * 128 + 64), 0, bar(B_FULL + sl));
        if (fmt_16bit(FMT)) {
          tma_load_2d(sa + off_phi, &tm_phi, static_cast<int32_t>(cb * 128), static_cast<int32_t>(rb * 128),
                      bar(B_FULL + sl));
          tma_load_2d(sa + off_phi + 16384u, &tm_phi, static_cast<int32_t>(cb * 128 + 64),
                      static_cast<int32_t>(rb * 128), bar(B_FULL + sl));
        } else {
          tma_load_2d(sa + off_phi, &tm_phi, static_cast<int32_t>(FMT == FMT_I4 ? cb * 64 : cb * 128),
                      static_cast<int32_t>(rb * 128), bar(B_FULL + sl));
        }
        pending = true, pend_sl = sl, pend_par = su & 1u;
        if (!(ok = wait_spin_bounded(bar(B_FULL + sl), su & 1u, ctl, 2))) break;
        pending = false;
        if (!(ok = wait_spin_bounded(bar(B_LEMPTY + b), (bu & 1u) ^ 1u, ctl, 3))) break;
        tc_fence_after();
        const uint64_t db = make_sdesc(sa + off_b, rbox, 1024, SWZ_128B);
        for (int ks = 0; ks < r16 / 16; ++ks) {
          const uint64_t da = AMN ? make_sdesc(sa + 2048u * ks, rbox, 1024, SWZ_128B)
                                  : make_sdesc(sa + 16384u * (ks >> 2) + 32u * (ks & 3), 16, 1024, SWZ_128B);
          mma_bf16(tmem + 128u * b, da, db + 128 * ks, idesc, ks > 0 ? 1u : 0u);
        }
        mma_commit(bar(B_LFULL + b));     // the low-rank tile is ready
      }
      // before the shared memory and TMEM are released: the last copy has landed and every
      // MMA has completed (already so unless a wait gave up)
      if (pending) drain_wait(bar(B_FULL + pend_sl), pend_par, args.timeout_ns);
      mma_commit(bar(B_DRAIN));
      drain_wait(bar(B_DRAIN), 0, args.timeout_ns);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    constexpr int NW = raw_words<FMT>();
    const QuantParams q = args.q;
    const uint32_t lr2 = pack_rn_bf16x2(q.lr_scale, q.lr_scale);   // exact: a power of two when UB
    const uint32_t lane_off = static_cast<uint32_t>(32 * warp) << 16;
    const uint32_t r_in = 32 * warp + lane;   // this thread's row inside a tile
    const uint32_t off_phi = a_tile_bytes(r16, AMN) + 2u * 128u * static_cast<uint32_t>(r16);
    const uint32_t sbytes = slot_bytes(r16, AMN, FMT);
    bool ok = true;
    uint32_t i = 0;
    for (int64_t t = blockIdx.x; t < num_tiles; t += gridDim.x, ++i) {
      const int64_t row = (t / nkb) * 128 + r_in;
      const int64_t colt = (t % nkb) * 128;
      const uint32_t b = i & 1u, bu = i >> 1, sl = i % nslot;
      const uint32_t phi_tile = smem + sl * sbytes + off_phi;
      // the tile's MMAs completed, so its operands (and base) are in the slot
      ok = wait_bounded(bar(B_LFULL + b), bu & 1u, ctl, 4);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        float v[32], L[32];
        uint32_t raw[NW];
        lds_raw32<FMT>(phi_tile, r_in, cc, raw);
        tmem_ld32(tmem + lane_off + 128u * b + 32u * cc, L);
        decode32<FMT>(raw, v);
        tmem_ld_wait();
        if (cc == 3) {
          // the tile's last reads of the slot and of the TMEM buffer: both may be refilled
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(bar(B_LEMPTY + b));
            mbar_arrive(bar(B_SEMPTY + sl));
          }
        }
        // t = u + magic rounds u half to even in units of 2^f; clamped to [lo, hi] its bit
        // pattern is the bits of magic (low byte zero) plus the integer code, so the code's
        // int8 two's complement is t's low byte (code_bias added: the biased code's byte).
        uint32_t o[8];
#pragma unroll
        for (int g = 0; g < 8; ++g) {
          uint32_t tb[4];
#pragma unroll
          for (int e = 0; e < 4; e += 2) {
            const int j = 4 * g + e;
            float2 tt;
            if (UB) {
              tt = __fadd2_rn(u_bf16x2(L[j], L[j + 1], v[j], v[j + 1], lr2), make_float2(q.magic, q.magic));
            } else {
              const float2 u = __ffma2_rn(make_float2(L[j], L[j + 1]), make_float2(q.lr_scale, q.lr_scale),
                                          make_float2(v[j], v[j + 1]));
              tt = __fadd2_rn(u, make_float2(q.magic, q.magic));
            }
            tb[e] = __float_as_uint(fminf(fmaxf(tt.x, q.lo), q.hi)) + args.code_bias;
            tb[e + 1] = __float_as_uint(fminf(fmaxf(tt.y, q.lo), q.hi)) + args.code_bias;
          }
          o[g] = __byte_perm(__byte_perm(tb[0], tb[1], 0x0040u), __byte_perm(tb[2], tb[3], 0x0040u), 0x5410u);
        }
        uint4* dst = reinterpret_cast<uint4*>(args.wz + row * args.k + colt + 32 * cc);
        dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
        dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == NUM_EPI_WARPS) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

template <int FMT, bool UB, bool AMN>
cudaError_t launch_merge_one(const CUtensorMap& tm_a, const CUtensorMap& tm_b, const CUtensorMap& tm_phi,
                             const MergeArgs& args, cudaStream_t stream) {
  static bool configured[kMaxDevices] = {};
  const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(merge_tc_kernel<FMT, UB, AMN>),
                                         static_cast<int>(MAX_SMEM_BYTES), configured);
  if (e != cudaSuccess) return e;
  static int sms[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e2 = cudaGetDevice(&dev);
  if (e2 != cudaSuccess) return e2;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (sms[dev] == 0) {
    e2 = cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev);
    if (e2 != cudaSuccess) return e2;
  }
  const int64_t tiles = (args.m / 128) * (args.k / 128);
  const uint32_t smem = smem_bytes(args.r16, AMN, FMT);
  const int64_t per_sm = 232448 / smem >= 2 ? 2 : 1;
  const int64_t grid = tiles < per_sm * sms[dev] ? tiles : per_sm * sms[dev];
  merge_tc_kernel<FMT, UB, AMN><<<static_cast<unsigned>(grid), NUM_THREADS, smem, stream>>>(tm_a, tm_b, tm_phi, args);
  return cudaGetLastError();
}

template <bool UB, bool AMN>
cudaError_t launch_merge_ub(int fmt, const CUtensorMap& tm_a, const CUtensorMap& tm_b, const CUtensorMap& tm_phi,
                            const MergeArgs& args,
                            cudaStream_t stream) {
  switch (fmt) {
    case FMT_Q8: return launch_merge_one<FMT_Q8, UB, AMN>(tm_a, tm_b, tm_phi, args, stream);
    case FMT_I4: return launch_merge_one<FMT_I4, UB, AMN>(tm_a, tm_b, tm_phi, args, stream);
    case FMT_BF16: return launch_merge_one<FMT_BF16, UB, AMN>(tm_a, tm_b, tm_phi, args, stream);
    case FMT_F16: return UB ? cudaErrorInvalidValue : launch_merge_one<FMT_F16, false, AMN>(tm_a, tm_b, tm_phi, args, stream);
    case FMT_E4M3: return launch_merge_one<FMT_E4M3, UB, AMN>(tm_a, tm_b, tm_phi, args, stream);
    case FMT_E5M2: return launch_merge_one<FMT_E5M2, UB, AMN>(tm_a, tm_b, tm_phi, args, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

static_assert(smem_bytes(256, true, FMT_BF16) <= MAX_SMEM_BYTES && smem_bytes(256, false, FMT_BF16) <= MAX_SMEM_BYTES,
              "smem budget");
static_assert(num_slots(32, true, FMT_Q8) == 3 && num_slots(256, true, FMT_BF16) == 1, "operand slots");

cudaError_t launch_merge_tc(int fmt, int u_bf16, int a_mn, const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const CUtensorMap& tm_phi, const MergeArgs& args, cudaStream_t stream) {
  if (args.m % 128 || args.k % 128 || args.r16 < 16 || args.r16 > 256 || (args.r16 & 15)) return cudaErrorInvalidValue;
  if (a_mn) return u_bf16 ? launch_merge_ub<true, true>(fmt, tm_a, tm_b, tm_phi, args, stream)
                          : launch_merge_ub<false, true>(fmt, tm_a, tm_b, tm_phi, args, stream);
  return u_bf16 ? launch_merge_ub<true, false>(fmt, tm_a, tm_b, tm_phi, args, stream)
                : launch_merge_ub<false, false>(fmt, tm_a, tm_b, tm_phi, args, stream);
}

}  // namespace lrqat
