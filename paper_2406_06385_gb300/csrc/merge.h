// Launcher of the tensor-core merge (merge.cu).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "quant.cuh"

namespace lrqat {

// W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p) on the tensor cores; A and B are read
// by TMA (tm_a over A [m, r], 64 x 128 boxes; tm_b over B [r, k], 64 x r16 boxes; both 128-byte
// swizzled), so r % 8 == 0 and both are 16-byte aligned, as are phi0 and wz.
struct MergeArgs {
  const void* phi0;      // stored base [m, k] in its format
  int8_t* wz;            // W_Z [m, k]
  int64_t m, k;
  int32_t r16;           // adapter rank rounded up to 16 (<= 64)
  QuantParams q;
  int* status;
  uint64_t timeout_ns;
};
// fmt: a PhiFmt value (quant.cuh); u_bf16: the bf16 pre-round value (not with FP16 bases)
cudaError_t launch_merge_tc(int fmt, int u_bf16, const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const MergeArgs& args, cudaStream_t stream);

}  // namespace lrqat
