// Launcher of the tensor-core low-rank code pass (merge.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "quant.cuh"

namespace lrqat {

// Codes clamp(round(phi^{-1}(Phi0) + (alpha/r) A B), lo, hi) of every element, int8, on the
// tensor cores.  With the quantizer's own [n, p] bounds in q this is the merge W_Z =
// clip(...) of Sec. 3; with [-128, 127] it is the unclipped code saturated to int8, which the
// GEMMs of ranks above 64 read as their base (the clip mask [n <= round(u) <= p] survives the
// saturation because n >= -64 and p <= 63 for b <= 7).
//   a_mn == 0: tm_a over A [m, r] (r % 8 == 0, 16-byte aligned), 64 x 128 boxes, K-major;
//   a_mn == 1: tm_a over the zero-padded A^T [r16, m], 64 x r16 boxes, MN-major.
//   tm_b over B [r, k] or the zero-padded B [r16, k], 64 x r16 boxes.  All 128-byte swizzled;
//   tm_phi over the stored base in 128-column chunks: 8-bit values 128 x 128 boxes (SW128),
//   packed nibbles 64-byte x 128-row boxes (SW64), 16-bit values 64 x 128 boxes (SW128);
//   wz 16-byte aligned.
struct MergeArgs {
  int8_t* wz;            // codes [m, k]
  int64_t m, k;
  int32_t r16;           // adapter rank rounded up to 16 (<= 256)
  QuantParams q;         // q.lo / q.hi: the clamp bounds in the magic domain
  int* status;
  uint64_t timeout_ns;
  uint32_t code_bias;    // added to every stored code: 0 (two's complement), 64 or 128 (c + bias, unsigned)
};
// fmt: a PhiFmt value (quant.cuh); u_bf16: the bf16 pre-round value (not with FP16 bases)
cudaError_t launch_merge_tc(int fmt, int u_bf16, int a_mn, const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const CUtensorMap& tm_phi, const MergeArgs& args, cudaStream_t stream);

}  // namespace lrqat
