// Internal launcher declarations shared by the translation units of liblrqat.
// Every launcher enqueues on `stream` and returns the cudaError_t of the launch.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "quant.cuh"

namespace lrqat {

// Devices a process may use with the library (ordinals 0 .. kMaxDevices - 1).
constexpr int kMaxDevices = 64;

// Raises a kernel's dynamic shared-memory limit to `bytes` on the current device,
// once per device: the attribute belongs to the device's context, so a process
// that uses several devices sets it on each.  `done` has kMaxDevices entries.
inline cudaError_t ensure_smem_attr(const void* kernel, int bytes, bool* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (!done[dev]) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  return cudaSuccess;
}

// ---- elementwise.cu --------------------------------------------------------
// z0 == nullptr: symmetric range setting (s0 only); else asymmetric (s0 and zero offsets z0).
cudaError_t launch_range_minmax(const float* W0, int64_t m, int64_t k, int group_size, int bits, float* s0,
                                float* z0, cudaStream_t stream);
// L^p range setting over N scaled min-max candidates (symmetric grids).
cudaError_t launch_range_lp(const float* W0, int64_t m, int64_t k, int group_size, int bits, float p_norm, int n_cand,
                            float* s0, cudaStream_t stream);
// fmt: a PhiFmt value (quant.cuh); zero offsets z0 only with the integer formats.
cudaError_t launch_downcast(const float* W0, const float* s0, const float* z0, int64_t m, int64_t k, int group_size,
                            int bits, int fmt, void* phi0, cudaStream_t stream);
cudaError_t launch_merge(const void* phi0, const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r,
                         int fmt, int u_bf16, const QuantParams& q, int8_t* wz, cudaStream_t stream);
// codes = clip(round(X / s_x), -128, 127) as bf16; optional mask bits [k][ceil(T/32)].
// Per-token dynamic int8 quantizer: s_x[t] = max |X[t, :]| / 127, writes
// X_hat = bf16(s_x[t] X_Z) [T, k].
cudaError_t launch_act_quant_token(const uint16_t* X, int64_t T, int64_t k, uint16_t* x_hat, cudaStream_t stream);
cudaError_t launch_act_quant(const uint16_t* X, int64_t T, int64_t k, const float* s_x, uint16_t* codes,
                             uint32_t* mask, cudaStream_t stream);
// TMA-friendly adapter layouts in one launch (null outputs are skipped):
// A_pad [m][64] = A zero-padded to 64 columns, Bt_pad [k][64] = B^T zero-padded,
// At [r16][m] = A^T with zero rows r..r16-1, B_pad [r16][k] = B with zero rows.
cudaError_t launch_adapter_layouts(const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r, int r16,
                                   uint16_t* A_pad, uint16_t* Bt_pad, uint16_t* At, uint16_t* B_pad,
                                   cudaStream_t stream);
// The backward's preparation in one launch: the adapter layouts (as launch_adapter_layouts)
// and phi_t[j][i] = stored value of Phi0[i][j]: the raw byte (Q-fixed, FP8), the
// sign-extended nibble as an int8 (packed INT-b), or the raw 16-bit pattern (BF16, FP16);
// phi_t [k, m].  clip_bits > 0 (int8 codes only): each value is clamped to the signed
// clip_bits-bit grid and biased by 64 on the way (the GEMMs' clip(c) + 64 codes).
cudaError_t launch_bwd_prep(const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r, int r16,
                            uint16_t* A_pad, uint16_t* Bt_pad, uint16_t* At, uint16_t* B_pad, const void* phi0,
                            int fmt, void* phi_t, cudaStream_t stream, int clip_bits = 0);
// Schedule of the dW work over its persistent CTAs.  The work is ni x nj tiles (128 rows i x
// 128 * nchunks columns j; tile = ib + ni * jt) of tsteps 32-token stages each; G and the
// gradients it feeds (dU, dA, dB, ds) are linear in the tokens, so any token range of a tile
// can be reduced on its own and its contribution written as one partial slot.
//   tail == 0: every tile is cut into nsplit equal token ranges (units), taken round robin.
//   tail == 1: the first full_tiles tiles (whole waves of `grid`) are taken whole, round robin,
//     so that the CTAs of a wave read the same token stages of neighbouring tiles; then CTA
//     b < tail_grid takes one part of a remaining tile: each of the tail_tiles tiles is cut into
//     tail_grid / tail_tiles or one more equal token ranges (parts j = 0, 1, ... write slots
//     j), so every CTA finishes one segment and the CTAs on neighbouring tiles start at the
//     same token offsets.  The dW kernel records each tile's part count in tile_segs for the
//     reduction.
struct DwSched {
  int32_t tail;
  int32_t grid;
  int64_t tsteps;        // stages of one tile: ceil(T / 32)
  int64_t full_tiles;    // tiles taken whole before the tail
  int64_t tail_tiles;    // tiles cut into parts (<= tail_grid)
  int64_t tail_grid;     // CTAs that take a tail part
};
// CTA b's tail part (b < tail_grid): tail tile t (tile full_tiles + t), part j of q.
__host__ __device__ inline void dw_tail_part(int64_t b, const DwSched& s, int64_t& t, int& j, int& q) {
  const int64_t q_lo = s.tail_grid / s.tail_tiles, extra = s.tail_grid % s.tail_tiles;
  const int64_t wide = extra * (q_lo + 1);   // CTAs of the tiles cut into q_lo + 1 parts
  if (b < wide) {
    t = b / (q_lo + 1);
    j = static_cast<int>(b % (q_lo + 1));
    q = static_cast<int>(q_lo + 1);
  } else {
    t = extra + (b - wide) / q_lo;
    j = static_cast<int>((b - wide) % q_lo);
    q = static_cast<int>(q_lo);
  }
}
// Partial slots a tile's segments write (tail == 1).
__host__ __device__ inline int dw_tile_segments(int64_t tile, const DwSched& s) {
  if (tile < s.full_tiles) return 1;
  const int64_t q_lo = s.tail_grid / s.tail_tiles, extra = s.tail_grid % s.tail_tiles;
  return static_cast<int>(tile - s.full_tiles < extra ? q_lo + 1 : q_lo);
}

// Deterministic sums of the per-tile gradient partials written by the dW kernel.
struct ReduceArgs {
  const float* dA_part; int nA;      // [nA][m][r]
  const float* dB_part; int nB;      // [nB][r][k]
  const float* ds_part; int nS;      // [nS][m][k/128]
  float* dA; float* dB; float* ds;
  int64_t m, k; int r; int group_size;
  float lr;                          // alpha / r
  int accumulate;
  // which partial slots hold data (all of them unless the dW work had a tail, sched.tail)
  DwSched sched;
  int ni, nsplit, bn;                // row blocks, slots per tile, columns per tile
  const int32_t* tile_segs;          // tail schedule: slots written per tile (by the dW kernel)
};
cudaError_t launch_reduce(const ReduceArgs& a, cudaStream_t stream);

// ---- optim.cu ----------------------------------------------------------------
cudaError_t launch_grad_sqnorm(const float* dA, int64_t na, const float* dB, int64_t nb, const float* ds, int64_t nc,
                               float* sqnorm, cudaStream_t stream);
struct AdamwArgs {
  const float* dA; const float* dB; const float* ds;
  float* A32; float* B32; float* s;
  float* mA; float* vA; float* mB; float* vB; float* ms; float* vs;
  uint16_t* A; uint16_t* B;          // bf16 copies of the updated A, B
  int64_t nA, nB, ns;
  float lr_ab, lr_s, wd_ab, wd_s;
  float beta1, beta2, eps, bc1, bc2;  // bc = 1 - beta^step
  float max_norm;
  const float* sqnorm;                // global squared gradient norm (device scalar)
};
cudaError_t launch_adamw(const AdamwArgs& a, cudaStream_t stream);

// ---- fused_gemm.cu ---------------------------------------------------------
enum FusedMode : int { FUSED_FWD_PC = 0, FUSED_FWD_GROUP = 1, FUSED_DX = 2 };

struct FusedArgs {
  int32_t rows;          // rows of the produced weight operand (m for fwd, k for dX)
  int32_t kdim;          // contraction length (k for fwd, m for dX)
  int32_t T;             // tokens
  int32_t r16;           // adapter rank rounded up to 16; 0: no low-rank term (the base holds
                         // the unclipped int8 codes round(u), written for ranks above 64)
  int32_t sf_cols;       // columns of the second factor loaded per stage (16, 32 or 64)
  int32_t num_rb;        // rows / 128
  int32_t num_tb;        // ceil(T / 448)
  int32_t num_tiles;
  QuantParams q;
  const float* s;        // scale, [m] or [m, s_ld]
  int32_t s_ld;          // groups per row (0 = per channel)
  int32_t group_size;
  const float* s_x;      // activation scale (device scalar) or nullptr
  const uint32_t* xmask; // dX only: activation clip mask bits [k][xmask_ld], or nullptr
  int32_t xmask_ld;
  uint16_t* out;         // Y [T, m] (fwd) or dX [T, k] (dX)
  int64_t out_ld;
  int* status;
  uint64_t timeout_ns;
  // Kept last: inserting it earlier shifted the fields above and slowed the producers.
  const float* zero;     // zero offsets shaped like s (asymmetric weights), or nullptr
  int32_t u_bf16;        // pre-round value in bf16 (lrqat_layer.u_bf16)
  // Forward only: the second factor's slice read straight from B as one MN-major box
  // of 64 columns x r16 rank rows (no padded B^T copy).
  int32_t sf_mn;
  // Codes base (r16 == 0): 0: saturated int8 codes (the producers clamp them); 64 or 128: the
  // codes clipped to [n, p] and stored as the unsigned byte c + 64 (b <= 7) or c + 128 (b = 8).
  int32_t codes_bias;
  // dX only: the scales (and zero offsets, or nullptr) as bf16 rows along the contraction,
  // [groups][kdim] (one row per channel scale), written by launch_dx_scales.
  const uint16_t* s_bf16;
  const uint16_t* z_bf16;
};
// s_out[g][i] = bf16(s[i][g]) (s [m] per channel: g = 0 only) and, with z, z_out likewise: the
// dX GEMM's producers read 16 consecutive of them per stage with two 16-byte loads.
cudaError_t launch_dx_scales(const float* s, const float* z, int64_t m, int groups, int s_ld, uint16_t* s_out,
                             uint16_t* z_out, cudaStream_t stream);
int fused_smem_bytes(int fmt);
// The same GEMM on CTA pairs (fused_pair.cu): 256-row x 448-token tiles, npairs clusters of 2.
// Needs rows % 256 == 0 and K-major factor slices (sf_mn == 0); tm_tok boxes of 112 tokens x
// 64, tm_sf boxes of 32 slice rows x sf_cols; tm_phi and tm_rf as for launch_fused.
cudaError_t launch_fused_pair(int mode, int fmt, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi,
                              const CUtensorMap& tm_rf, const CUtensorMap& tm_sf, const FusedArgs& args, int npairs,
                              cudaStream_t stream);
// fmt: a PhiFmt value (quant.cuh); FMT_I4 only for the forward modes
cudaError_t launch_fused(int mode, int fmt, const CUtensorMap& tm_tok, const CUtensorMap& tm_phi,
                         const CUtensorMap& tm_rf, const CUtensorMap& tm_sf, const FusedArgs& args, int grid,
                         cudaStream_t stream);

// ---- dw.cu -------------------------------------------------------------------
struct DwArgs {
  int32_t m, k, T;
  int32_t r, r16;
  int32_t nchunks;       // 128-column chunks per tile (1 or 2)
  int32_t ni, nj, nsplit, tchunk, num_units;
  QuantParams q;
  const float* s; int32_t s_ld; int32_t group_size;
  const float* s_x;
  float* dA_part; float* dB_part; float* ds_part;
  int* status;
  uint64_t timeout_ns;
  const float* zero;     // zero offsets shaped like s (asymmetric weights), or nullptr
  const void* phi;       // 16-bit bases only: Phi0 [m, k], read directly by the epilogue
  int32_t u_bf16;        // pre-round value in bf16 (lrqat_layer.u_bf16)
  DwSched sched;         // kept last (argument layout)
  int32_t* tile_segs;    // tail schedule: [ni * nj] slots written per tile
  // Ranks above 64: the base (tm_phi) holds the unclipped int8 codes round(u), low-rank
  // term included; no low-rank tile, nchunks == 1, tm_at / tm_b boxes of 64 rank rows.
  int32_t codes_base;
};
int dw_smem_bytes(int r16, int fmt);
// The same kernel on CTA pairs (dw_pair.cu) for ranks up to 64, m and k multiples of 256:
// units of 256 x 256 tiles (args.ni = m / 256, args.nj = k / 256, nchunks 2), npairs clusters of
// two; tm_ath / tm_bh as tm_at / tm_b with boxes of r16 / 2 rank rows.  The partials are laid out
// as launch_dw's (dB per 128-row block, tile_segs per 128-row tile).
cudaError_t launch_dw_pair(int fmt, const CUtensorMap& tm_dy, const CUtensorMap& tm_x, const CUtensorMap& tm_at,
                           const CUtensorMap& tm_ath, const CUtensorMap& tm_phi, const CUtensorMap& tm_b,
                           const CUtensorMap& tm_bh, const DwArgs& args, int npairs, cudaStream_t stream);
// Clusters of two of the pair dW kernel that can be resident at once on the current device
// (0 when the query fails).
int dw_pair_max_pairs();
// fmt: a PhiFmt value (quant.cuh)
cudaError_t launch_dw(int fmt, const CUtensorMap& tm_dy, const CUtensorMap& tm_x, const CUtensorMap& tm_at,
                      const CUtensorMap& tm_phi, const CUtensorMap& tm_b, const DwArgs& args, int grid,
                      cudaStream_t stream);

}  // namespace lrqat
