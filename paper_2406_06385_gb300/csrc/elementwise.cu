// Memory-bound kernels of the LR-QAT layer: range setting, downcast (Eq. 6/7),
// merge into integer weights (Sec. 3, after Eq. 8), the per-tensor int8
// activation quantizer, operand re-layouts for the fused GEMMs, and the
// deterministic reduction of per-tile gradient partials.
#include <cuda_runtime.h>
#include <cstdint>

#include "kernels.h"
#include "quant.cuh"

namespace lrqat {
namespace {

constexpr int kThreads = 256;

inline int blocks_for(int64_t n, int per_block) {
  int64_t b = (n + per_block - 1) / per_block;
  return static_cast<int>(b > 0x7FFFFFFF ? 0x7FFFFFFF : b);
}

// ------------------------------------------------------------ range setting --
// One block per (row, group): s0 = max|W0| / p over the segment (1 if all zero).
__global__ void range_minmax_kernel(const float* __restrict__ W0, int64_t k, int seg, int ngroups, float p,
                                    float* __restrict__ s0) {
  const int64_t row = blockIdx.x / ngroups;
  const int g = blockIdx.x % ngroups;
  const float* src = W0 + row * k + static_cast<int64_t>(g) * seg;
  float amax = 0.0f;
  for (int j = threadIdx.x; j < seg; j += blockDim.x) amax = fmaxf(amax, fabsf(src[j]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  __shared__ float warp_max[kThreads / 32];
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = amax;
  __syncthreads();
  if (threadIdx.x == 0) {
    float a = 0.0f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) a = fmaxf(a, warp_max[w]);
    s0[blockIdx.x] = a > 0.0f ? __fdiv_rn(a, p) : 1.0f;
  }
}

// ----------------------------------------------------------------- downcast --
// Q-fixed (Eq. 7): round(2^f clip(W0/s0, n, p)) -> int8; 4 elements per thread.
__global__ void downcast_qfixed_kernel(const float4* __restrict__ W0, const float* __restrict__ s0, int64_t k,
                                       int group_size, int ngroups, float n, float p, float two_f,
                                       char4* __restrict__ out, int64_t n4) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n4;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = (e * 4) / k;
    const int64_t col = (e * 4) % k;
    const float s = group_size ? s0[row * ngroups + col / group_size] : s0[row];
    const float4 w = W0[e];
    const float x[4] = {w.x, w.y, w.z, w.w};
    int q[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float y = fminf(fmaxf(__fdiv_rn(x[i], s), n), p) * two_f;   // exact scaling by 2^f
      q[i] = __float2int_rn(y);
    }
    out[e] = make_char4(static_cast<signed char>(q[0]), static_cast<signed char>(q[1]),
                        static_cast<signed char>(q[2]), static_cast<signed char>(q[3]));
  }
}

// INT-b, double packed: clip(round(W0/s0), n, p), two nibbles per byte; 8 elements per thread.
__global__ void downcast_packed_kernel(const float4* __restrict__ W0, const float* __restrict__ s0, int64_t k,
                                       int group_size, int ngroups, int n, int p, uint32_t* __restrict__ out,
                                       int64_t n8) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n8;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = (e * 8) / k;
    const int64_t col = (e * 8) % k;
    const float s = group_size ? s0[row * ngroups + col / group_size] : s0[row];
    const float4 w0 = W0[2 * e];
    const float4 w1 = W0[2 * e + 1];
    const float x[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
    uint32_t word = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      int c = __float2int_rn(__fdiv_rn(x[i], s));
      c = c < n ? n : (c > p ? p : c);
      word |= (static_cast<uint32_t>(c) & 0xFu) << (4 * i);
    }
    out[e] = word;
  }
}

// -------------------------------------------------------------------- merge --
// W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p); A B by fp32 FMAs over t = 0..r-1.
constexpr int kMergeRows = 16;
__global__ void merge_kernel(const void* __restrict__ phi0, const uint16_t* __restrict__ A,
                             const uint16_t* __restrict__ B, int64_t m, int64_t k, int r, int packed, QuantParams q,
                             int8_t* __restrict__ wz) {
  __shared__ float As[kMergeRows][64];
  const int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  const int64_t i0 = static_cast<int64_t>(blockIdx.y) * kMergeRows;
  for (int e = threadIdx.x; e < kMergeRows * 64; e += blockDim.x) {
    const int ii = e / 64, t = e % 64;
    As[ii][t] = (i0 + ii < m && t < r) ? bf16_to_float(A[(i0 + ii) * r + t]) : 0.0f;
  }
  __syncthreads();
  if (j >= k) return;
  float bcol[64];
#pragma unroll
  for (int t = 0; t < 64; ++t) bcol[t] = t < r ? bf16_to_float(B[static_cast<int64_t>(t) * k + j]) : 0.0f;
  for (int ii = 0; ii < kMergeRows && i0 + ii < m; ++ii) {
    const int64_t i = i0 + ii;
    float L = 0.0f;
#pragma unroll
    for (int t = 0; t < 64; ++t)
      if (t < r) L = __fmaf_rn(As[ii][t], bcol[t], L);
    float v;
    if (packed) {
      const uint8_t byte = static_cast<const uint8_t*>(phi0)[i * (k / 2) + j / 2];
      int nib = (j & 1) ? (byte >> 4) : (byte & 0xF);
      v = static_cast<float>(nib >= 8 ? nib - 16 : nib);
    } else {
      v = static_cast<float>(static_cast<const int8_t*>(phi0)[i * k + j]);
    }
    wz[i * k + j] = static_cast<int8_t>(__float2int_rn(lrqat_code(L, v, q)));
  }
}

// --------------------------------------------------------- activation quant --
// X_Z = clip(round(X / s_x), -128, 127) stored as exact bf16; optional mask bits
// M_x = 1[-128 <= round(X / s_x) <= 127], laid out [k][ceil(T/32)] (bit = token % 32).
__global__ void act_quant_kernel(const uint16_t* __restrict__ X, int64_t T, int64_t k, const float* __restrict__ s_x,
                                 uint16_t* __restrict__ codes, uint32_t* __restrict__ mask, int64_t mask_ld) {
  const int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (j >= k) return;
  const float sx = *s_x;
  const int64_t t0 = static_cast<int64_t>(blockIdx.y) * 32;
  uint32_t word = 0;
  for (int tt = 0; tt < 32; ++tt) {
    const int64_t t = t0 + tt;
    if (t >= T) break;
    const float x = bf16_to_float(X[t * k + j]);
    const float qv = rintf(__fdiv_rn(x, sx));
    const float c = fminf(fmaxf(qv, -128.0f), 127.0f);
    codes[t * k + j] = static_cast<uint16_t>(__float_as_uint(c) >> 16);
    if (qv >= -128.0f && qv <= 127.0f) word |= 1u << tt;
  }
  if (mask) mask[j * mask_ld + blockIdx.y] = word;
}

// ---------------------------------------------------------------- re-layouts --
__global__ void pad_rows64_kernel(const uint16_t* __restrict__ A, int64_t m, int r, uint16_t* __restrict__ out) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= m * 64) return;
  const int64_t i = e / 64;
  const int c = static_cast<int>(e % 64);
  out[e] = c < r ? A[i * r + c] : static_cast<uint16_t>(0);
}

__global__ void pad_rows_kernel(const uint16_t* __restrict__ src, int rows, int rows_pad, int64_t cols,
                                uint16_t* __restrict__ out) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= static_cast<int64_t>(rows_pad) * cols) return;
  const int c = static_cast<int>(e / cols);
  out[e] = c < rows ? src[e] : static_cast<uint16_t>(0);
}

__global__ void transpose_pad64_kernel(const uint16_t* __restrict__ B, int r, int64_t k, uint16_t* __restrict__ out) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= k * 64) return;
  const int64_t j = e / 64;
  const int c = static_cast<int>(e % 64);
  out[e] = c < r ? B[static_cast<int64_t>(c) * k + j] : static_cast<uint16_t>(0);
}

__global__ void transpose_rows_kernel(const uint16_t* __restrict__ A, int64_t m, int r, int r16,
                                      uint16_t* __restrict__ out) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= static_cast<int64_t>(r16) * m) return;
  const int c = static_cast<int>(e / m);
  const int64_t i = e % m;
  out[e] = c < r ? A[i * r + c] : static_cast<uint16_t>(0);
}

// 64 x 64 tiles of Phi0 (rows i, columns j) -> out[j][i] as int8 stored integers.
__global__ void phi_transpose_kernel(const void* __restrict__ phi0, int64_t m, int64_t k, int packed,
                                     int8_t* __restrict__ out) {
  __shared__ int8_t tile[64][64 + 4];
  const int64_t i0 = static_cast<int64_t>(blockIdx.y) * 64;
  const int64_t j0 = static_cast<int64_t>(blockIdx.x) * 64;
  for (int e = threadIdx.x; e < 64 * 64; e += blockDim.x) {
    const int ii = e / 64, jj = e % 64;
    const int64_t i = i0 + ii, j = j0 + jj;
    int8_t v;
    if (packed) {
      const uint8_t byte = static_cast<const uint8_t*>(phi0)[i * (k / 2) + j / 2];
      const int nib = (j & 1) ? (byte >> 4) : (byte & 0xF);
      v = static_cast<int8_t>(nib >= 8 ? nib - 16 : nib);
    } else {
      v = static_cast<const int8_t*>(phi0)[i * k + j];
    }
    tile[ii][jj] = v;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 64 * 64; e += blockDim.x) {
    const int jj = e / 64, ii = e % 64;
    out[(j0 + jj) * m + i0 + ii] = tile[ii][jj];
  }
}

// ------------------------------------------------------------------- reduce --
__global__ void reduce_rows_kernel(const float* __restrict__ part, int nparts, int64_t n, float lr, int accumulate,
                                   float* __restrict__ dst) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n) return;
  float acc = 0.0f;
  for (int p = 0; p < nparts; ++p) acc += part[static_cast<int64_t>(p) * n + e];
  acc *= lr;
  dst[e] = accumulate ? dst[e] + acc : acc;
}

__global__ void reduce_ds_kernel(const float* __restrict__ part, int nparts, int64_t m, int64_t nb, int ngroups,
                                 int blocks_per_group, int accumulate, float* __restrict__ ds) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= m * ngroups) return;
  const int64_t i = e / ngroups;
  const int g = static_cast<int>(e % ngroups);
  float acc = 0.0f;
  for (int p = 0; p < nparts; ++p) {
    const float* row = part + (static_cast<int64_t>(p) * m + i) * nb;
    for (int b = g * blocks_per_group; b < (g + 1) * blocks_per_group; ++b) acc += row[b];
  }
  ds[e] = accumulate ? ds[e] + acc : acc;
}

}  // namespace

cudaError_t launch_range_minmax(const float* W0, int64_t m, int64_t k, int group_size, int p, float* s0,
                                cudaStream_t stream) {
  const int ngroups = group_size ? static_cast<int>(k / group_size) : 1;
  const int seg = group_size ? group_size : static_cast<int>(k);
  range_minmax_kernel<<<static_cast<unsigned>(m * ngroups), kThreads, 0, stream>>>(W0, k, seg, ngroups,
                                                                                   static_cast<float>(p), s0);
  return cudaGetLastError();
}

cudaError_t launch_downcast(const float* W0, const float* s0, int64_t m, int64_t k, int group_size, int bits,
                            int packed, void* phi0, cudaStream_t stream) {
  const int ngroups = group_size ? static_cast<int>(k / group_size) : 1;
  const int n = -(1 << (bits - 1)), p = (1 << (bits - 1)) - 1;
  if (!packed) {
    const int64_t n4 = m * k / 4;
    downcast_qfixed_kernel<<<blocks_for(n4, kThreads), kThreads, 0, stream>>>(
        reinterpret_cast<const float4*>(W0), s0, k, group_size, ngroups, static_cast<float>(n),
        static_cast<float>(p), static_cast<float>(1 << (8 - bits)), static_cast<char4*>(phi0), n4);
  } else {
    const int64_t n8 = m * k / 8;
    downcast_packed_kernel<<<blocks_for(n8, kThreads), kThreads, 0, stream>>>(
        reinterpret_cast<const float4*>(W0), s0, k, group_size, ngroups, n, p, static_cast<uint32_t*>(phi0), n8);
  }
  return cudaGetLastError();
}

cudaError_t launch_merge(const void* phi0, const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r,
                         int packed, const QuantParams& q, int8_t* wz, cudaStream_t stream) {
  dim3 grid(static_cast<unsigned>((k + kThreads - 1) / kThreads), static_cast<unsigned>((m + kMergeRows - 1) / kMergeRows));
  merge_kernel<<<grid, kThreads, 0, stream>>>(phi0, A, B, m, k, r, packed, q, wz);
  return cudaGetLastError();
}

cudaError_t launch_act_quant(const uint16_t* X, int64_t T, int64_t k, const float* s_x, uint16_t* codes,
                             uint32_t* mask, cudaStream_t stream) {
  dim3 grid(static_cast<unsigned>((k + 127) / 128), static_cast<unsigned>((T + 31) / 32));
  act_quant_kernel<<<grid, 128, 0, stream>>>(X, T, k, s_x, codes, mask, (T + 31) / 32);
  return cudaGetLastError();
}

cudaError_t launch_pad_rows64(const uint16_t* A, int64_t m, int r, uint16_t* out, cudaStream_t stream) {
  pad_rows64_kernel<<<blocks_for(m * 64, kThreads), kThreads, 0, stream>>>(A, m, r, out);
  return cudaGetLastError();
}

cudaError_t launch_pad_rows(const uint16_t* src, int rows, int rows_pad, int64_t cols, uint16_t* out,
                            cudaStream_t stream) {
  pad_rows_kernel<<<blocks_for(static_cast<int64_t>(rows_pad) * cols, kThreads), kThreads, 0, stream>>>(src, rows, rows_pad,
                                                                                                      cols, out);
  return cudaGetLastError();
}

cudaError_t launch_transpose_pad64(const uint16_t* B, int r, int64_t k, uint16_t* out, cudaStream_t stream) {
  transpose_pad64_kernel<<<blocks_for(k * 64, kThreads), kThreads, 0, stream>>>(B, r, k, out);
  return cudaGetLastError();
}

cudaError_t launch_transpose_rows(const uint16_t* A, int64_t m, int r, int r16, uint16_t* out,
                                  cudaStream_t stream) {
  transpose_rows_kernel<<<blocks_for(static_cast<int64_t>(r16) * m, kThreads), kThreads, 0, stream>>>(A, m, r, r16,
                                                                                                     out);
  return cudaGetLastError();
}

cudaError_t launch_phi_transpose(const void* phi0, int64_t m, int64_t k, int packed, int8_t* out,
                                 cudaStream_t stream) {
  dim3 grid(static_cast<unsigned>(k / 64), static_cast<unsigned>(m / 64));
  phi_transpose_kernel<<<grid, kThreads, 0, stream>>>(phi0, m, k, packed, out);
  return cudaGetLastError();
}

cudaError_t launch_reduce(const ReduceArgs& a, cudaStream_t stream) {
  const int64_t nA = a.m * a.r, nB = static_cast<int64_t>(a.r) * a.k;
  reduce_rows_kernel<<<blocks_for(nA, kThreads), kThreads, 0, stream>>>(a.dA_part, a.nA, nA, a.lr, a.accumulate, a.dA);
  reduce_rows_kernel<<<blocks_for(nB, kThreads), kThreads, 0, stream>>>(a.dB_part, a.nB, nB, a.lr, a.accumulate, a.dB);
  const int64_t nb = a.k / 128;
  const int ngroups = a.group_size ? static_cast<int>(a.k / a.group_size) : 1;
  const int bpg = a.group_size ? a.group_size / 128 : static_cast<int>(nb);
  reduce_ds_kernel<<<blocks_for(a.m * ngroups, kThreads), kThreads, 0, stream>>>(a.ds_part, a.nS, a.m, nb, ngroups,
                                                                                bpg, a.accumulate, a.ds);
  return cudaGetLastError();
}

}  // namespace lrqat
