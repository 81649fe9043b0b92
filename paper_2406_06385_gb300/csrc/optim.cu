// Optimizer step on the trainable parameters of an LR-QAT layer (App. B, Table B1):
// AdamW with decoupled weight decay over A, B (fp32 master copies, bf16 copies for the
// GEMMs) and the scales s, after clipping the global L2 norm of all trainable
// gradients.  The norm is accumulated layer by layer into one device scalar.
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int kNormThreads = 1024;

// Sum of squares of dA, dB and ds, added into *sqnorm.  One block: each thread adds a
// fixed strided subset in order (fp64), then a fixed tree adds the threads, so the
// result does not depend on scheduling.
__global__ void __launch_bounds__(kNormThreads) grad_sqnorm_kernel(const float* __restrict__ a, int64_t na,
                                                                   const float* __restrict__ b, int64_t nb,
                                                                   const float* __restrict__ c, int64_t nc,
                                                                   float* __restrict__ sqnorm) {
  double acc = 0.0;
  for (int64_t i = threadIdx.x; i < na; i += kNormThreads) acc += static_cast<double>(a[i]) * a[i];
  for (int64_t i = threadIdx.x; i < nb; i += kNormThreads) acc += static_cast<double>(b[i]) * b[i];
  for (int64_t i = threadIdx.x; i < nc; i += kNormThreads) acc += static_cast<double>(c[i]) * c[i];
  __shared__ double part[kNormThreads];
  part[threadIdx.x] = acc;
  __syncthreads();
  for (int h = kNormThreads / 2; h > 0; h >>= 1) {
    if (static_cast<int>(threadIdx.x) < h) part[threadIdx.x] += part[threadIdx.x + h];
    __syncthreads();
  }
  if (threadIdx.x == 0) *sqnorm = static_cast<float>(static_cast<double>(*sqnorm) + part[0]);
}

struct AdamSeg {
  const float* g;     // gradient
  float* p;           // fp32 parameter (master copy)
  float* m;
  float* v;
  uint16_t* p_bf16;   // bf16 copy written after the update, or nullptr
  int64_t n;
  float lr, wd;
};

// One AdamW step per element of three segments (A, B, s) in one launch:
//   g <- coef g;  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2;
//   p <- p (1 - lr wd) - lr (m / bc1) / (sqrt(v / bc2) + eps)
// with coef = min(1, max_norm / (sqrt(sqnorm) + 1e-6)) (1 when max_norm <= 0).
__global__ void adamw_kernel(AdamSeg s0, AdamSeg s1, AdamSeg s2, const float* __restrict__ sqnorm, float max_norm,
                             float beta1, float beta2, float eps, float bc1, float bc2) {
  const float coef = max_norm > 0.0f ? fminf(1.0f, max_norm / (sqrtf(*sqnorm) + 1e-6f)) : 1.0f;
  const int64_t total = s0.n + s1.n + s2.n;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const AdamSeg& S = e < s0.n ? s0 : (e < s0.n + s1.n ? s1 : s2);
    const int64_t i = e < s0.n ? e : (e < s0.n + s1.n ? e - s0.n : e - s0.n - s1.n);
    const float g = coef * S.g[i];
    const float m = beta1 * S.m[i] + (1.0f - beta1) * g;
    const float v = beta2 * S.v[i] + (1.0f - beta2) * g * g;
    S.m[i] = m;
    S.v[i] = v;
    const float p = S.p[i] * (1.0f - S.lr * S.wd) - S.lr * (m / bc1) / (sqrtf(v / bc2) + eps);
    S.p[i] = p;
    if (S.p_bf16) S.p_bf16[i] = static_cast<uint16_t>(pack_rn_bf16x2(p, 0.0f) & 0xFFFFu);
  }
}

}  // namespace

cudaError_t launch_grad_sqnorm(const float* dA, int64_t na, const float* dB, int64_t nb, const float* ds, int64_t nc,
                               float* sqnorm, cudaStream_t stream) {
  grad_sqnorm_kernel<<<1, kNormThreads, 0, stream>>>(dA, na, dB, nb, ds, nc, sqnorm);
  return cudaGetLastError();
}

cudaError_t launch_adamw(const AdamwArgs& a, cudaStream_t stream) {
  const AdamSeg s0{a.dA, a.A32, a.mA, a.vA, a.A, a.nA, a.lr_ab, a.wd_ab};
  const AdamSeg s1{a.dB, a.B32, a.mB, a.vB, a.B, a.nB, a.lr_ab, a.wd_ab};
  const AdamSeg s2{a.ds, a.s, a.ms, a.vs, nullptr, a.ns, a.lr_s, a.wd_s};
  const int64_t total = a.nA + a.nB + a.ns;
  const int64_t want = (total + 255) / 256;
  const unsigned grid = static_cast<unsigned>(want < 2048 ? want : 2048);
  adamw_kernel<<<grid, 256, 0, stream>>>(s0, s1, s2, a.sqnorm, a.max_norm, a.beta1, a.beta2, a.eps, a.bc1, a.bc2);
  return cudaGetLastError();
}

}  // namespace lrqat
