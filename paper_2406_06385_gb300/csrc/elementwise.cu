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

// Asymmetric min-max range setting (zero offsets, Eq. 1): per (row, group)
// s0 = (max - min) / (2^b - 1) in fp32 (1 if max == min) and
// z0 = clip(round(n - min / s0), n, p), min / s0 one fp32 division, the rest exact.
__global__ void range_minmax_asym_kernel(const float* __restrict__ W0, int64_t k, int seg, int ngroups, int bits,
                                         float* __restrict__ s0, float* __restrict__ z0) {
  const int64_t row = blockIdx.x / ngroups;
  const int g = blockIdx.x % ngroups;
  const float* src = W0 + row * k + static_cast<int64_t>(g) * seg;
  float lo = INFINITY, hi = -INFINITY;
  for (int j = threadIdx.x; j < seg; j += blockDim.x) {
    const float v = src[j];
    lo = fminf(lo, v);
    hi = fmaxf(hi, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  __shared__ float warp_lo[kThreads / 32], warp_hi[kThreads / 32];
  if ((threadIdx.x & 31) == 0) {
    warp_lo[threadIdx.x >> 5] = lo;
    warp_hi[threadIdx.x >> 5] = hi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) {
      lo = fminf(lo, warp_lo[w]);
      hi = fmaxf(hi, warp_hi[w]);
    }
    const float span = __fsub_rn(hi, lo);
    const float s = span > 0.0f ? __fdiv_rn(span, static_cast<float>((1 << bits) - 1)) : 1.0f;
    const double n = -static_cast<double>(1 << (bits - 1)), p = static_cast<double>((1 << (bits - 1)) - 1);
    const double z = fmin(fmax(rint(n - static_cast<double>(__fdiv_rn(lo, s))), n), p);
    s0[blockIdx.x] = s;
    z0[blockIdx.x] = static_cast<float>(z);
  }
}

// ----------------------------------------------------------------- downcast --
// Q-fixed (Eq. 7): round(2^f clip(W0/s0, n, p)) -> int8; 4 elements per thread.
// With zero offsets z0 (nullable): round(2^f clip(W0/s0 + z0, n, p)), the integer
// offset added exactly in double precision.
__global__ void downcast_qfixed_kernel(const float4* __restrict__ W0, const float* __restrict__ s0,
                                       const float* __restrict__ z0, int64_t k, int group_size, int ngroups,
                                       float n, float p, float two_f, char4* __restrict__ out, int64_t n4) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n4;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = (e * 4) / k;
    const int64_t col = (e * 4) % k;
    const int64_t sidx = group_size ? row * ngroups + col / group_size : row;
    const float s = s0[sidx];
    const float4 w = W0[e];
    const float x[4] = {w.x, w.y, w.z, w.w};
    int q[4];
    if (z0 == nullptr) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float y = fminf(fmaxf(__fdiv_rn(x[i], s), n), p) * two_f;   // exact scaling by 2^f
        q[i] = __float2int_rn(y);
      }
    } else {
      const double z = z0[sidx];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const double y = fmin(fmax(static_cast<double>(__fdiv_rn(x[i], s)) + z, static_cast<double>(n)),
                              static_cast<double>(p)) * two_f;
        q[i] = __double2int_rn(y);
      }
    }
    out[e] = make_char4(static_cast<signed char>(q[0]), static_cast<signed char>(q[1]),
                        static_cast<signed char>(q[2]), static_cast<signed char>(q[3]));
  }
}

// INT-b, double packed: clip(round(W0/s0), n, p), two nibbles per byte; 8 elements per thread.
// With zero offsets z0 (nullable): clip(round(W0/s0 + z0), n, p).
__global__ void downcast_packed_kernel(const float4* __restrict__ W0, const float* __restrict__ s0,
                                       const float* __restrict__ z0, int64_t k, int group_size, int ngroups, int n,
                                       int p, uint32_t* __restrict__ out, int64_t n8) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n8;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = (e * 8) / k;
    const int64_t col = (e * 8) % k;
    const int64_t sidx = group_size ? row * ngroups + col / group_size : row;
    const float s = s0[sidx];
    const double z = z0 != nullptr ? static_cast<double>(z0[sidx]) : 0.0;
    const float4 w0 = W0[2 * e];
    const float4 w1 = W0[2 * e + 1];
    const float x[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
    uint32_t word = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      int c = z0 == nullptr ? __float2int_rn(__fdiv_rn(x[i], s))
                            : __double2int_rn(static_cast<double>(__fdiv_rn(x[i], s)) + z);
      c = c < n ? n : (c > p ? p : c);
      word |= (static_cast<uint32_t>(c) & 0xFu) << (4 * i);
    }
    out[e] = word;
  }
}

// Floating-point storage (Sec. 3, the cast choices of phi): Phi0 = cast(fl32(W0 / s0))
// with round-to-nearest-even, no clipping inside phi, FP16 and FP8 saturating at their
// largest finite value; 4 elements per thread.
template <int FMT>
__device__ __forceinline__ uint32_t pack_fp8x2(float lo, float hi) {
  unsigned short r;
  if (FMT == FMT_E4M3) asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  else asm("cvt.rn.satfinite.e5m2x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// Saturating: values beyond 65504 (which round-to-nearest would turn into infinities)
// are clamped to it first.
__device__ __forceinline__ uint32_t pack_sat_f16x2(float lo, float hi) {
  uint32_t r;
  lo = fminf(fmaxf(lo, -65504.0f), 65504.0f);
  hi = fminf(fmaxf(hi, -65504.0f), 65504.0f);
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

template <int FMT>
__global__ void downcast_float_kernel(const float4* __restrict__ W0, const float* __restrict__ s0, int64_t k,
                                      int group_size, int ngroups, void* __restrict__ out, int64_t n4) {
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n4;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t row = (e * 4) / k;
    const int64_t col = (e * 4) % k;
    const float s = s0[group_size ? row * ngroups + col / group_size : row];
    const float4 w = W0[e];
    const float x0 = __fdiv_rn(w.x, s), x1 = __fdiv_rn(w.y, s), x2 = __fdiv_rn(w.z, s), x3 = __fdiv_rn(w.w, s);
    if (FMT == FMT_BF16) {
      static_cast<uint2*>(out)[e] = make_uint2(pack_rn_bf16x2(x0, x1), pack_rn_bf16x2(x2, x3));
    } else if (FMT == FMT_F16) {
      static_cast<uint2*>(out)[e] = make_uint2(pack_sat_f16x2(x0, x1), pack_sat_f16x2(x2, x3));
    } else {
      static_cast<uint32_t*>(out)[e] = pack_fp8x2<FMT>(x0, x1) | (pack_fp8x2<FMT>(x2, x3) << 16);
    }
  }
}

// 4 stored values of a row -> phi^{-1}(Phi0) in the units of u_f (Eq. 7 / Eq. 8).
__device__ __forceinline__ void decode_row4(const void* phi0, int64_t i, int64_t k, int64_t j, int fmt, float* v) {
  if (fmt == FMT_I4) {
    // 4 columns = 2 packed bytes (low nibble = even column)
    const uint16_t two = *reinterpret_cast<const uint16_t*>(static_cast<const uint8_t*>(phi0) + i * (k / 2) + j / 2);
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int nib = (two >> (4 * c)) & 0xF;
      v[c] = static_cast<float>(nib >= 8 ? nib - 16 : nib);
    }
  } else if (fmt_16bit(fmt)) {
    const uint2 w = *reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(phi0) + i * k + j);
    if (fmt == FMT_BF16) {
      decode_16x2_raw<FMT_BF16>(w.x, v);
      decode_16x2_raw<FMT_BF16>(w.y, v + 2);
    } else {
      decode_16x2_raw<FMT_F16>(w.x, v);
      decode_16x2_raw<FMT_F16>(w.y, v + 2);
#pragma unroll
      for (int c = 0; c < 4; ++c) v[c] *= kFloatRebias<FMT_F16>;
    }
  } else {
    const uint32_t four = *reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(phi0) + i * k + j);
    if (fmt == FMT_Q8) {
#pragma unroll
      for (int c = 0; c < 4; ++c) v[c] = static_cast<float>(static_cast<int8_t>((four >> (8 * c)) & 0xFF));
    } else if (fmt == FMT_E4M3) {
      decode_fp8x4_raw<FMT_E4M3>(four, v);
#pragma unroll
      for (int c = 0; c < 4; ++c) v[c] *= kFloatRebias<FMT_E4M3>;
    } else {
      decode_fp8x4_raw<FMT_E5M2>(four, v);
#pragma unroll
      for (int c = 0; c < 4; ++c) v[c] *= kFloatRebias<FMT_E5M2>;
    }
  }
}

// -------------------------------------------------------------------- merge --
// W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p).  Each thread owns a
// register tile of 16 rows x 4 columns: per rank index t it reads 16 values of A
// (shared memory, broadcast) and 4 of B, and does 64 FMAs, so the product A B runs
// at FMA throughput; the 4 codes of a row go out as one 32-bit store.
constexpr int kMergeRows = 16;
constexpr int kMergeThreads = 128;
constexpr int kMergeCols = 4 * kMergeThreads;   // 512 columns per block
__global__ void __launch_bounds__(kMergeThreads) merge_kernel(const void* __restrict__ phi0,
                                                              const uint16_t* __restrict__ A,
                                                              const uint16_t* __restrict__ B, int64_t m, int64_t k,
                                                              int r, int fmt, int ub, int b_aligned, QuantParams q,
                                                              int8_t* __restrict__ wz) {
  __shared__ __align__(16) float As[64][kMergeRows];   // A^T tile of 64 rank indices: [t][row]
  const int64_t i0 = static_cast<int64_t>(blockIdx.y) * kMergeRows;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * kMergeCols + 4 * threadIdx.x;
  float acc[kMergeRows][4];
#pragma unroll
  for (int ii = 0; ii < kMergeRows; ++ii)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[ii][c] = 0.0f;
  // the rank in blocks of 64 indices, A staged in shared memory per block
  for (int t0 = 0; t0 < r; t0 += 64) {
  __syncthreads();   // the previous block's reads of As are done
  for (int e = threadIdx.x; e < kMergeRows * 64; e += kMergeThreads) {
    const int t = e / kMergeRows, ii = e % kMergeRows;
    As[t][ii] = (i0 + ii < m && t0 + t < r) ? bf16_to_float(A[(i0 + ii) * r + t0 + t]) : 0.0f;
  }
  __syncthreads();
  if (j < k) {
  const int t_end = r - t0 < 64 ? r - t0 : 64;
  for (int tt = 0; tt < t_end; ++tt) {
    const int t = t0 + tt;
    const uint16_t* brow = B + static_cast<int64_t>(t) * k + j;
    uint2 braw;
    if (b_aligned) {
      braw = __ldg(reinterpret_cast<const uint2*>(brow));
    } else {
      braw.x = static_cast<uint32_t>(brow[0]) | (static_cast<uint32_t>(brow[1]) << 16);
      braw.y = static_cast<uint32_t>(brow[2]) | (static_cast<uint32_t>(brow[3]) << 16);
    }
    const float b4[4] = {__uint_as_float(braw.x << 16), __uint_as_float(braw.x & 0xFFFF0000u),
                         __uint_as_float(braw.y << 16), __uint_as_float(braw.y & 0xFFFF0000u)};
    const float4* arow = reinterpret_cast<const float4*>(&As[tt][0]);
#pragma unroll
    for (int g = 0; g < kMergeRows / 4; ++g) {
      const float4 a4 = arow[g];
      const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[4 * g + u][c] = __fmaf_rn(av[u], b4[c], acc[4 * g + u][c]);
    }
  }
  }
  }
  if (j >= k) return;
#pragma unroll
  for (int ii = 0; ii < kMergeRows; ++ii) {
    const int64_t i = i0 + ii;
    if (i >= m) break;
    float v[4];
    decode_row4(phi0, i, k, j, fmt, v);
    if (ub) {
      // bf16 pre-round value: u_f = bf16(v + bf16(lr_f bf16(L))); the code of an exact u_f
      const uint32_t lr2 = pack_rn_bf16x2(q.lr_scale, q.lr_scale);
#pragma unroll
      for (int c = 0; c < 4; c += 2) {
        const float2 u = u_bf16x2(acc[ii][c], acc[ii][c + 1], v[c], v[c + 1], lr2);
        v[c] = u.x;
        v[c + 1] = u.y;
        acc[ii][c] = 0.0f;
        acc[ii][c + 1] = 0.0f;
      }
    }
    uint32_t out = 0;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int code = __float2int_rn(lrqat_code(acc[ii][c], v[c], q));
      out |= (static_cast<uint32_t>(code) & 0xFFu) << (8 * c);
    }
    *reinterpret_cast<uint32_t*>(wz + i * k + j) = out;
  }
}

// round(fl(x / s)) with fl the IEEE fp32 division, without dividing in the common
// case: y = x * r with r = fl(1 / s) is within |y| 2^-22 of x / s, and fl(x / s) within
// |y| 2^-24, so unless y lies within |y| 2^-20 (+ a tiny absolute margin) of a
// half-integer both round to the same integer; near a half-integer the exact
// division decides.
__device__ __forceinline__ float div_round(float x, float s, float r) {
  const float y = x * r;
  const float q = rintf(y);
  if (fabsf(fabsf(y - q) - 0.5f) > fmaxf(fabsf(y), 1.0f) * 9.5367431640625e-07f) return q;   // 2^-20
  return rintf(__fdiv_rn(x, s));
}

// --------------------------------------------------------- activation quant --
// round(fl32(x / s)) for two values, dividing only near a tie: y = x r with r =
// fl32(1 / s) lies within 2^-22 |y| of x / s, and so does fl32(x / s); for |y| < 2^10
// that is below 2^-12, so a y more than 2^-11 away from a half-integer rounds like the
// exact quotient.  A |y| >= 2^10 is far outside every grid quantized here (|code| <=
// 128), so whichever integer it rounds to, it clips and masks the same way.
__device__ __forceinline__ float2 div_round2(float2 x, float s, float r) {
  const float2 y = __fmul2_rn(x, make_float2(r, r));
  float2 q = make_float2(rintf(y.x), rintf(y.y));
  const float2 d = __fadd2_rn(y, make_float2(-q.x, -q.y));
  if (fabsf(d.x) > 0.49951171875f) q.x = rintf(__fdiv_rn(x.x, s));
  if (fabsf(d.y) > 0.49951171875f) q.y = rintf(__fdiv_rn(x.y, s));
  return q;
}

// round(fl32(x / s)) for the 8 bf16 values of a 16-byte word, with one near-tie test for
// all of them (the largest distance from a half-integer decides whether any needs the
// IEEE division); same results as div_round2 on each pair.
__device__ __forceinline__ void div_round8(const uint4& raw, float s, float r, float (&q)[8]) {
  const uint32_t in[4] = {raw.x, raw.y, raw.z, raw.w};
  float x[8], dmax = 0.0f;
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    x[2 * h] = __uint_as_float(in[h] << 16);
    x[2 * h + 1] = __uint_as_float(in[h] & 0xFFFF0000u);
    const float2 y = __fmul2_rn(make_float2(x[2 * h], x[2 * h + 1]), make_float2(r, r));
    q[2 * h] = rintf(y.x);
    q[2 * h + 1] = rintf(y.y);
    const float2 d = __fadd2_rn(y, make_float2(-q[2 * h], -q[2 * h + 1]));
    dmax = fmaxf(dmax, fmaxf(fabsf(d.x), fabsf(d.y)));
  }
  if (dmax > 0.49951171875f) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float y = x[e] * r;
      if (fabsf(y - q[e]) > 0.49951171875f) q[e] = rintf(__fdiv_rn(x[e], s));
    }
  }
}

// Per-tensor quantizer: X_Z = clip(round(X / s_x), -128, 127) stored as exact bf16;
// optional mask bits M_x = 1[-128 <= round(X / s_x) <= 127], laid out [k][ceil(T/32)]
// (bit = token % 32).  A block covers 64 columns x 256 tokens; lane (colgroup =
// lane / 4, token group g = lane % 4) of warp w handles 8 columns (16 bytes) of tokens
// 32w + 8g .. + 7, so one load instruction covers four token rows of 128 contiguous
// bytes, and a lane issues its 8 loads before it uses any.  The mask bytes gather in
// shared memory, and each column's 8 words (256 tokens) go out as 32 contiguous bytes.
// (A persistent grid that loads its next tile while quantizing the current one held
// only two blocks per SM and ran slower.)
constexpr int kAqWarps = 8;
constexpr int kAqTokens = 32 * kAqWarps;
__global__ void __launch_bounds__(32 * kAqWarps) act_quant_kernel(const uint4* __restrict__ X, int64_t T,
                                                                  int64_t k8, const float* __restrict__ s_x,
                                                                  uint4* __restrict__ codes,
                                                                  uint32_t* __restrict__ mask, int64_t mask_ld) {
  __shared__ __align__(16) uint8_t mbytes[64][4 * kAqWarps];   // [column][token byte]
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int cg = lane >> 2, g = lane & 3;
  const int64_t c8 = static_cast<int64_t>(blockIdx.x) * 8 + cg;
  const int64_t t0 = static_cast<int64_t>(blockIdx.y) * kAqTokens + 32 * w + 8 * g;
  const bool col_ok = c8 < k8;
  const float sx = *s_x;
  const float rx = __frcp_rn(sx);
  uint4 v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
    v[i] = col_ok && t0 + i < T ? __ldg(X + (t0 + i) * k8 + c8) : make_uint4(0u, 0u, 0u, 0u);
  uint32_t bits[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (col_ok && t0 + i < T) {
      float q[8];
      div_round8(v[i], sx, rx, q);
      uint32_t out[4];
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const float c0 = fminf(fmaxf(q[2 * h], -128.0f), 127.0f), c1 = fminf(fmaxf(q[2 * h + 1], -128.0f), 127.0f);
        out[h] = pack_rn_bf16x2(c0, c1);
        bits[2 * h] |= static_cast<uint32_t>(c0 == q[2 * h]) << i;       // in range iff the clip kept it
        bits[2 * h + 1] |= static_cast<uint32_t>(c1 == q[2 * h + 1]) << i;
      }
      codes[(t0 + i) * k8 + c8] = make_uint4(out[0], out[1], out[2], out[3]);
    }
  }
  if (mask == nullptr) return;
#pragma unroll
  for (int e = 0; e < 8; ++e) mbytes[8 * cg + e][4 * w + g] = static_cast<uint8_t>(bits[e]);
  __syncthreads();
  // 64 columns x 8 words: thread -> column tid / 4, words 2 (tid % 4), + 1
  const int col = threadIdx.x >> 2, q = threadIdx.x & 3;
  const int64_t j = static_cast<int64_t>(blockIdx.x) * 64 + col;
  const int64_t w0 = static_cast<int64_t>(blockIdx.y) * kAqWarps + 2 * q;
  if (j < 8 * k8) {
    const uint2 pair = *reinterpret_cast<const uint2*>(&mbytes[col][8 * q]);
    uint32_t* dst = mask + j * mask_ld + w0;
    if (w0 + 1 < mask_ld && ((reinterpret_cast<uintptr_t>(dst) & 7u) == 0)) {
      *reinterpret_cast<uint2*>(dst) = pair;
    } else {
      if (w0 < mask_ld) dst[0] = pair.x;
      if (w0 + 1 < mask_ld) dst[1] = pair.y;
    }
  }
}

// Per-token dynamic int8 quantizer: s_x[t] = max_j |X[t, j]| / 127 (1 for an all-zero
// token), X_Z = clip(round(X / s_x[t]), -128, 127) with the IEEE division, and X_hat =
// bf16(s_x[t] X_Z), the operand of the forward and dW GEMMs.  A token gets 2^tpt_log2
// threads (32 .. 256, at most kAtLoads 16-byte loads each: k <= 16384), which keep its
// row in registers from the absmax pass to the quantize pass, so the row is read from
// memory once; a block of 256 threads holds 256 >> tpt_log2 tokens.  Absmax scaling
// never clips, so no mask is needed.
constexpr int kAtLoads = 8;
__global__ void __launch_bounds__(256, 3) act_quant_token_kernel(const uint4* __restrict__ X, int64_t T, int64_t k8,
                                                                 int tpt_log2, uint4* __restrict__ out) {
  __shared__ float red[8];
  const int tpt = 1 << tpt_log2;
  const int sub = threadIdx.x & (tpt - 1);                        // thread within its token
  const int64_t t = static_cast<int64_t>(blockIdx.x) * (256 >> tpt_log2) + (threadIdx.x >> tpt_log2);
  const bool live = t < T;
  const uint4* row = X + (live ? t : 0) * k8;
  uint4 v[kAtLoads];
#pragma unroll
  for (int i = 0; i < kAtLoads; ++i) {
    const int64_t j = sub + static_cast<int64_t>(tpt) * i;
    v[i] = live && j < k8 ? __ldg(row + j) : make_uint4(0u, 0u, 0u, 0u);
  }
  float amax = 0.0f;
#pragma unroll
  for (int i = 0; i < kAtLoads; ++i) {
    const uint32_t in[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
    for (int h = 0; h < 4; ++h)
      amax = fmaxf(amax, fmaxf(fabsf(__uint_as_float(in[h] << 16)), fabsf(__uint_as_float(in[h] & 0xFFFF0000u))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  if (tpt > 32) {   // the warps of one token combine through shared memory
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
    __syncthreads();
    const int w0 = (threadIdx.x >> 5) & ~((tpt >> 5) - 1);
    for (int w = 0; w < (tpt >> 5); ++w) amax = fmaxf(amax, red[w0 + w]);
  }
  if (!live) return;
  const float sx = amax > 0.0f ? __fdiv_rn(amax, 127.0f) : 1.0f;
  const float rx = __frcp_rn(sx);
#pragma unroll
  for (int i = 0; i < kAtLoads; ++i) {
    const int64_t j = sub + static_cast<int64_t>(tpt) * i;
    if (j < k8) {
      // absmax scaling: |X / s_x| <= 127 (+ rounding), so the codes need no clip
      float q[8];
      div_round8(v[i], sx, rx, q);
      uint32_t o[4];
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const float2 xh = __fmul2_rn(make_float2(q[2 * h], q[2 * h + 1]), make_float2(sx, sx));
        o[h] = pack_rn_bf16x2(xh.x, xh.y);
      }
      out[t * k8 + j] = make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
}

// The same for rows longer than the register-resident kernel holds (k > 16384): one
// warp per token, the second pass rereads the row.
__global__ void __launch_bounds__(kThreads) act_quant_token_wide_kernel(const uint4* __restrict__ X, int64_t T,
                                                                        int64_t k8, uint4* __restrict__ out) {
  const int64_t t = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const uint4* row = X + t * k8;
  float amax = 0.0f;
  for (int64_t j = lane; j < k8; j += 32) {
    const uint4 v = row[j];
    const uint32_t in[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int h = 0; h < 4; ++h)
      amax = fmaxf(amax, fmaxf(fabsf(__uint_as_float(in[h] << 16)), fabsf(__uint_as_float(in[h] & 0xFFFF0000u))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float sx = amax > 0.0f ? __fdiv_rn(amax, 127.0f) : 1.0f;
  const float rx = __frcp_rn(sx);
  for (int64_t j = lane; j < k8; j += 32) {
    const uint4 v = row[j];
    const uint32_t in[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const float2 q =
          div_round2(make_float2(__uint_as_float(in[h] << 16), __uint_as_float(in[h] & 0xFFFF0000u)), sx, rx);
      const float2 xh = __fmul2_rn(make_float2(fminf(fmaxf(q.x, -128.0f), 127.0f), fminf(fmaxf(q.y, -128.0f), 127.0f)),
                                   make_float2(sx, sx));
      o[h] = pack_rn_bf16x2(xh.x, xh.y);
    }
    out[t * k8 + j] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// L^p range setting (symmetric), one block per (row, group): the segment is staged in
// shared memory, s_max = max|w| / p as in min-max, and thread j < N evaluates the
// candidate s_j = fl32(s_max (j + 1) / N): loss_j = sum |w - s_j clip(round(w / s_j), n, p)|^p
// (w / s_j decided as one fp32 division, the error formed with one fused multiply-add,
// |err|^p by multiplication for integer p).  The smallest loss wins, the smaller j on
// a tie.
__global__ void __launch_bounds__(kThreads) range_lp_kernel(const float* __restrict__ W0, int64_t k, int seg,
                                                            int ngroups, int bits, float p_norm, int n_cand,
                                                            float* __restrict__ s0) {
  extern __shared__ float segw[];
  const int64_t row = blockIdx.x / ngroups;
  const int g = blockIdx.x % ngroups;
  const float* src = W0 + row * k + static_cast<int64_t>(g) * seg;
  float amax = 0.0f;
  for (int j = threadIdx.x; j < seg; j += blockDim.x) {
    const float v = src[j];
    segw[j] = v;
    amax = fmaxf(amax, fabsf(v));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  __shared__ float warp_max[kThreads / 32];
  __shared__ float best_loss[kThreads];
  __shared__ int best_j[kThreads];
  if ((threadIdx.x & 31) == 0) warp_max[threadIdx.x >> 5] = amax;
  __syncthreads();
  float a = 0.0f;
  for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) a = fmaxf(a, warp_max[w]);
  const float pmax = static_cast<float>((1 << (bits - 1)) - 1), nmin = -static_cast<float>(1 << (bits - 1));
  const float s_max = a > 0.0f ? __fdiv_rn(a, pmax) : 1.0f;
  const int j = threadIdx.x;
  float loss = INFINITY;
  if (j < n_cand) {
    const float s = static_cast<float>(static_cast<double>(s_max) * (j + 1) / n_cand);
    const float r = __frcp_rn(s);
    const int ip = static_cast<int>(p_norm);
    const bool int_p = static_cast<float>(ip) == p_norm && ip >= 1 && ip <= 8;
    float acc0 = 0.0f, acc1 = 0.0f;
    for (int e = 0; e < seg; ++e) {
      const float w = segw[e];
      const float q = fminf(fmaxf(div_round(w, s, r), nmin), pmax);
      const float err = fabsf(fmaf(-s, q, w));
      float t;
      if (int_p) {
        t = err;
        for (int i = 1; i < ip; ++i) t *= err;
      } else {
        t = err > 0.0f ? powf(err, p_norm) : 0.0f;
      }
      if (e & 1) acc1 += t; else acc0 += t;
    }
    loss = acc0 + acc1;
  }
  best_loss[threadIdx.x] = loss;
  best_j[threadIdx.x] = j;
  __syncthreads();
  for (int h = blockDim.x / 2; h > 0; h >>= 1) {
    if (static_cast<int>(threadIdx.x) < h) {
      const float lo = best_loss[threadIdx.x + h];
      const int jo = best_j[threadIdx.x + h];
      if (lo < best_loss[threadIdx.x] || (lo == best_loss[threadIdx.x] && jo < best_j[threadIdx.x])) {
        best_loss[threadIdx.x] = lo;
        best_j[threadIdx.x] = jo;
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) s0[blockIdx.x] = static_cast<float>(static_cast<double>(s_max) * (best_j[0] + 1) / n_cand);
}

// ---------------------------------------------------------------- re-layouts --
// The four TMA-friendly layouts of the adapters, in one launch; each thread writes
// 8 consecutive bf16 (16 bytes) of one output.  Null outputs are skipped.
//   A_pad  [m][64]   = A[i][c], zero for c >= r       (row factor of the forward)
//   Bt_pad [k][64]   = B[c][j], zero for c >= r       (B^T, row factor of dX)
//   At     [r16][m]  = A[i][c], zero rows for c >= r  (A^T, dW epilogue)
//   B_pad  [r16][k]  = B[c][j], zero rows for c >= r  (dW epilogue)
__device__ __forceinline__ void adapter_layouts_body(int64_t blk, int64_t nblk, const uint16_t* __restrict__ A, const uint16_t* __restrict__ B, int64_t m,
                                       int64_t k, int r, int r16, uint4* __restrict__ A_pad,
                                       uint4* __restrict__ Bt_pad, uint4* __restrict__ At,
                                       uint4* __restrict__ B_pad, int b_aligned) {
  const int64_t n0 = A_pad ? m * 8 : 0;
  const int64_t n1 = Bt_pad ? k * 8 : 0;
  const int64_t n2 = At ? static_cast<int64_t>(r16) * (m / 8) : 0;
  const int64_t n3 = B_pad ? static_cast<int64_t>(r16) * (k / 8) : 0;
  const int64_t total = n0 + n1 + n2 + n3;
  for (int64_t t = blk * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < total;
       t += nblk * blockDim.x) {
    uint32_t w[4];
    if (t < n0) {
      const int64_t i = t >> 3;
      const int c0 = static_cast<int>(t & 7) * 8;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int c = c0 + 2 * e;
        const uint32_t lo = c < r ? A[i * r + c] : 0u, hi = c + 1 < r ? A[i * r + c + 1] : 0u;
        w[e] = lo | (hi << 16);
      }
      A_pad[t] = make_uint4(w[0], w[1], w[2], w[3]);
    } else if (t < n0 + n1) {
      const int64_t u = t - n0, j = u >> 3;
      const int c0 = static_cast<int>(u & 7) * 8;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int c = c0 + 2 * e;
        const uint32_t lo = c < r ? B[static_cast<int64_t>(c) * k + j] : 0u;
        const uint32_t hi = c + 1 < r ? B[static_cast<int64_t>(c + 1) * k + j] : 0u;
        w[e] = lo | (hi << 16);
      }
      Bt_pad[u] = make_uint4(w[0], w[1], w[2], w[3]);
    } else if (t < n0 + n1 + n2) {
      const int64_t u = t - n0 - n1;
      const int c = static_cast<int>(u / (m / 8));
      const int64_t i0 = (u % (m / 8)) * 8;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t lo = c < r ? A[(i0 + 2 * e) * r + c] : 0u, hi = c < r ? A[(i0 + 2 * e + 1) * r + c] : 0u;
        w[e] = lo | (hi << 16);
      }
      At[u] = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
      const int64_t u = t - n0 - n1 - n2;
      const int c = static_cast<int>(u / (k / 8));
      const int64_t j0 = (u % (k / 8)) * 8;
      if (c >= r) {
        B_pad[u] = make_uint4(0, 0, 0, 0);
      } else if (b_aligned) {
        B_pad[u] = *reinterpret_cast<const uint4*>(B + static_cast<int64_t>(c) * k + j0);
      } else {
        const uint16_t* src = B + static_cast<int64_t>(c) * k + j0;
#pragma unroll
        for (int e = 0; e < 4; ++e) w[e] = static_cast<uint32_t>(src[2 * e]) | (static_cast<uint32_t>(src[2 * e + 1]) << 16);
        B_pad[u] = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
}
__global__ void adapter_layouts_kernel(const uint16_t* __restrict__ A, const uint16_t* __restrict__ B, int64_t m,
                                       int64_t k, int r, int r16, uint4* __restrict__ A_pad,
                                       uint4* __restrict__ Bt_pad, uint4* __restrict__ At,
                                       uint4* __restrict__ B_pad, int b_aligned) {
  adapter_layouts_body(blockIdx.x, gridDim.x, A, B, m, k, r, r16, A_pad, Bt_pad, At, B_pad, b_aligned);
}

// 128 x 128 tiles of Phi0 (rows i, columns j) -> out[j][i] as int8 stored integers.
// Load: each thread brings four pieces of 16 stored integers (16 bytes, or 8 packed
// bytes) into a shared tile whose 16-byte groups are XOR-swizzled by the row's
// 16-row block, so that the column gathers below hit 32 distinct banks.
// Store: each thread transposes a 16-row x 4-column block with byte permutes and
// writes four 16-byte pieces of transposed rows (8 threads cover one 128-byte row).
__device__ __forceinline__ void unpack_i4x8(uint32_t packed4, uint32_t& lo_word, uint32_t& hi_word) {
  // 4 packed bytes -> 8 sign-extended nibbles (low nibble = even column)
  const uint32_t x = packed4 ^ 0x88888888u;
  const uint32_t lo = x & 0x0F0F0F0Fu, hi = (x >> 4) & 0x0F0F0F0Fu;
  lo_word = __vsub4(__byte_perm(lo, hi, 0x5140), 0x08080808u);
  hi_word = __vsub4(__byte_perm(lo, hi, 0x7362), 0x08080808u);
}

// clip_lo/clip_hi (clip != 0): int8 codes are clamped to [clip_lo, clip_hi] (each byte of the
// word the same bound) and biased by 64 on the way, for a consumer that reads clip(c) + 64.
__device__ __forceinline__ void phi_transpose_body(int64_t bx, int64_t by, const void* __restrict__ phi0, int64_t m, int64_t k,
                                                             int packed, int8_t* __restrict__ out, int clip = 0,
                                                             uint32_t clip_lo = 0, uint32_t clip_hi = 0) {
  __shared__ __align__(16) uint32_t tile[128 * 32];   // 128 rows x 32 words
  const int64_t i0 = by * 128;
  const int64_t j0 = bx * 128;
  const int t = threadIdx.x;
  uint4 v[4];
  if (packed) {
    const uint8_t* src = static_cast<const uint8_t*>(phi0);
    uint2 raw[4];
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const int u = t + 256 * x, R = u >> 3, q = u & 7;
      raw[x] = *reinterpret_cast<const uint2*>(src + (i0 + R) * (k / 2) + (j0 + 16 * q) / 2);
    }
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      unpack_i4x8(raw[x].x, v[x].x, v[x].y);
      unpack_i4x8(raw[x].y, v[x].z, v[x].w);
    }
  } else {
    const int8_t* src = static_cast<const int8_t*>(phi0);
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const int u = t + 256 * x, R = u >> 3, q = u & 7;
      v[x] = *reinterpret_cast<const uint4*>(src + (i0 + R) * k + j0 + 16 * q);
    }
    if (clip) {
      // per byte: max, min (signed), then + 64 without carries between bytes
      auto cb = [&](uint32_t w) { return __vadd4(__vmins4(__vmaxs4(w, clip_lo), clip_hi), 0x40404040u); };
#pragma unroll
      for (int x = 0; x < 4; ++x) v[x] = make_uint4(cb(v[x].x), cb(v[x].y), cb(v[x].z), cb(v[x].w));
    }
  }
#pragma unroll
  for (int x = 0; x < 4; ++x) {
    const int u = t + 256 * x, R = u >> 3, q = u & 7;
    *reinterpret_cast<uint4*>(&tile[R * 32 + 4 * (q ^ ((R >> 4) & 7))]) = v[x];
  }
  __syncthreads();
  const int w = t >> 5, L = t & 31;
  const int a = L & 7;                    // 16-row block of the tile (rows i)
  const int c = 4 * w + (L >> 3);         // word column: columns j = 4c .. 4c + 3
  const int wcol = 4 * (w ^ a) + (L >> 3);   // its swizzled position (all rows of block a)
  uint32_t o[4][4];
#pragma unroll
  for (int blk = 0; blk < 4; ++blk) {
    const int R = 16 * a + 4 * blk;
    const uint32_t x0 = tile[R * 32 + wcol], x1 = tile[(R + 1) * 32 + wcol];
    const uint32_t x2 = tile[(R + 2) * 32 + wcol], x3 = tile[(R + 3) * 32 + wcol];
    const uint32_t t01lo = __byte_perm(x0, x1, 0x5140), t01hi = __byte_perm(x0, x1, 0x7362);
    const uint32_t t23lo = __byte_perm(x2, x3, 0x5140), t23hi = __byte_perm(x2, x3, 0x7362);
    o[0][blk] = __byte_perm(t01lo, t23lo, 0x5410);
    o[1][blk] = __byte_perm(t01lo, t23lo, 0x7632);
    o[2][blk] = __byte_perm(t01hi, t23hi, 0x5410);
    o[3][blk] = __byte_perm(t01hi, t23hi, 0x7632);
  }
#pragma unroll
  for (int r = 0; r < 4; ++r)
    *reinterpret_cast<uint4*>(out + (j0 + 4 * c + r) * m + i0 + 16 * a) = make_uint4(o[r][0], o[r][1], o[r][2], o[r][3]);
}

// 16-bit bases: out[j][i] = Phi0[i][j] through a padded 64 x 64 shared tile (a row
// stride of 33 words keeps the column reads free of bank conflicts).
__device__ __forceinline__ void phi_transpose16_body(int64_t bx, int64_t by, const uint16_t* __restrict__ in, int64_t m, int64_t k,
                                                               uint16_t* __restrict__ out) {
  __shared__ __align__(16) uint32_t tile[64 * 33];   // 64 rows x 64 values (+ 2 values of padding)
  const int64_t i0 = by * 64;
  const int64_t j0 = bx * 64;
  const int t = threadIdx.x;
#pragma unroll
  for (int x = 0; x < 2; ++x) {
    const int u = t + 256 * x, R = u >> 3, q = u & 7;
    const uint4 v = *reinterpret_cast<const uint4*>(in + (i0 + R) * k + j0 + 8 * q);
    uint32_t* dst = &tile[R * 33 + 4 * q];
    dst[0] = v.x, dst[1] = v.y, dst[2] = v.z, dst[3] = v.w;
  }
  __syncthreads();
  const uint16_t* t16 = reinterpret_cast<const uint16_t*>(tile);
#pragma unroll
  for (int x = 0; x < 2; ++x) {
    const int u = t + 256 * x, J = u >> 3, q = u & 7;   // output row j0 + J, values i0 + 8q .. + 7
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e)
      o[e] = static_cast<uint32_t>(t16[(8 * q + 2 * e) * 66 + J]) |
             (static_cast<uint32_t>(t16[(8 * q + 2 * e + 1) * 66 + J]) << 16);
    *reinterpret_cast<uint4*>(out + (j0 + J) * m + i0 + 8 * q) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// The backward's preparation in one launch: blocks [0, n_layout) write the adapter
// layouts (as adapter_layouts_kernel), the rest transpose the stored base (as the
// 128 x 128 byte or 64 x 64 sixteen-bit transposes), one tile per block.
struct LayoutJob {
  const uint16_t* A; const uint16_t* B; int64_t m, k; int r, r16;
  uint4* A_pad; uint4* Bt_pad; uint4* At; uint4* B_pad; int b_aligned;
};
struct TransposeJob {
  const void* phi0; void* out; int64_t m, k; int fmt; int64_t nbx;   // tiles along k
  int clip; uint32_t clip_lo, clip_hi;   // int8 codes: clamp to [lo, hi] and add 64 (bytes x4)
};
__global__ void __launch_bounds__(256) bwd_prep_kernel(LayoutJob lj, int64_t n_layout, TransposeJob tj) {
  if (static_cast<int64_t>(blockIdx.x) < n_layout) {
    adapter_layouts_body(blockIdx.x, n_layout, lj.A, lj.B, lj.m, lj.k, lj.r, lj.r16, lj.A_pad, lj.Bt_pad, lj.At,
                         lj.B_pad, lj.b_aligned);
    return;
  }
  const int64_t b = blockIdx.x - n_layout;
  if (fmt_16bit(tj.fmt)) {
    phi_transpose16_body(b % tj.nbx, b / tj.nbx, static_cast<const uint16_t*>(tj.phi0), tj.m, tj.k,
                         static_cast<uint16_t*>(tj.out));
  } else {
    phi_transpose_body(b % tj.nbx, b / tj.nbx, tj.phi0, tj.m, tj.k, tj.fmt == FMT_I4, static_cast<int8_t*>(tj.out),
                       tj.clip, tj.clip_lo, tj.clip_hi);
  }
}

// ------------------------------------------------------------------- reduce --
// One launch sums every gradient partial. Block ranges: [0, nblk_a) dA, then dB, then ds.
// dA / dB: a block owns 32 float4 columns; warp w adds parts w, w + 8, w + 16, ... in that
// order, and the eight warp sums are added in a fixed tree, so results are deterministic.
constexpr int kRedSlices = kThreads / 32;

struct RedJob {
  const float4* part;
  int nparts;
  int64_t n4;
  float4* dst;
  int kind;        // 0: dA [m][r] (slot p = jt * nsplit + sp), 1: dB [r][k] (p = ib * nsplit + sp)
  int64_t width;   // r (dA) or k (dB): elements per row of a partial
};

// Whether partial slot sp of tile (ib, jt) was written by the dW kernel: every slot, unless
// its schedule had a tail (then a tail tile has as many slots as parts, which the dW kernel
// recorded).
__device__ __forceinline__ bool slot_written(const ReduceArgs& a, int64_t ib, int64_t jt, int sp) {
  if (!a.sched.tail || sp == 0) return true;
  const int64_t tile = ib + a.ni * jt;
  return tile >= a.sched.full_tiles && sp < __ldg(a.tile_segs + tile);
}

__device__ __forceinline__ void add4(float4& a, const float4& b) {
  a.x += b.x;
  a.y += b.y;
  a.z += b.z;
  a.w += b.w;
}

__device__ __forceinline__ void reduce_parts_block(const RedJob& j, int64_t blk, const ReduceArgs& a,
                                                   float4 (*sm)[32]) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t e = blk * 32 + lane;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  auto part = [&](int64_t p) { return __ldg(j.part + p * j.n4 + e); };
  if (e < j.n4 && !a.sched.tail) {
    int p = w;
    for (; p + 3 * kRedSlices < j.nparts; p += 4 * kRedSlices) {
      const float4 v0 = part(p);
      const float4 v1 = part(p + kRedSlices);
      const float4 v2 = part(p + 2 * kRedSlices);
      const float4 v3 = part(p + 3 * kRedSlices);
      add4(acc, v0);
      add4(acc, v1);
      add4(acc, v2);
      add4(acc, v3);
    }
    for (; p < j.nparts; p += kRedSlices) add4(acc, part(p));
  } else if (e < j.n4) {
    // With a tail: slot 0 of every tile (always written), spread over the warps, then the further
    // slots of the tail's tiles.  Slot p = o * nsplit + sp, o the other tile coordinate (jt for
    // dA, ib for dB); the tile coordinate this element fixes is the same for the whole block.
    const int ns = a.nsplit;
    const int64_t n_other = j.nparts / ns;
    const int64_t fixed = j.kind == 0 ? (4 * e / j.width) / 128 : ((4 * e) % j.width) / a.bn;
    // first o whose tile (fixed + ni o for dA, o + ni fixed for dB) is past the whole tiles;
    // this warp's first tail tile's part count is requested before the slot-0 loads
    const int64_t ft = a.sched.full_tiles;
    const int64_t o_tail = j.kind == 0 ? (ft > fixed ? (ft - fixed + a.ni - 1) / a.ni : 0)
                                       : (ft > a.ni * fixed ? ft - a.ni * fixed : 0);
    auto tile_of = [&](int64_t oo) { return j.kind == 0 ? fixed + a.ni * oo : oo + a.ni * fixed; };
    int segs0 = o_tail + w < n_other ? __ldg(a.tile_segs + tile_of(o_tail + w)) : 0;
    int64_t o = w;
    for (; o + 3 * kRedSlices < n_other; o += 4 * kRedSlices) {
      const float4 v0 = part(o * ns);
      const float4 v1 = part((o + kRedSlices) * ns);
      const float4 v2 = part((o + 2 * kRedSlices) * ns);
      const float4 v3 = part((o + 3 * kRedSlices) * ns);
      add4(acc, v0);
      add4(acc, v1);
      add4(acc, v2);
      add4(acc, v3);
    }
#pragma unroll 4
    for (; o < n_other; o += kRedSlices) add4(acc, part(o * ns));
    for (int64_t o2 = o_tail + w; o2 < n_other; o2 += kRedSlices) {
      const int segs = segs0;
      if (o2 + kRedSlices < n_other) segs0 = __ldg(a.tile_segs + tile_of(o2 + kRedSlices));
      // slots 1 .. segs - 1, four loads in flight at a time
      for (int sp = 1; sp < segs; sp += 4) {
        float4 v[4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
          v[q] = sp + q < segs ? part(o2 * ns + sp + q) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int q = 0; q < 4; ++q) add4(acc, v[q]);
      }
    }
  }
  sm[w][lane] = acc;
  __syncthreads();
  if (w == 0 && e < j.n4) {
    float4 s[kRedSlices];
#pragma unroll
    for (int i = 0; i < kRedSlices; ++i) s[i] = sm[i][lane];
#pragma unroll
    for (int h = kRedSlices / 2; h > 0; h >>= 1)
#pragma unroll
      for (int i = 0; i < h; ++i) add4(s[i], s[i + h]);
    float4 r = make_float4(s[0].x * a.lr, s[0].y * a.lr, s[0].z * a.lr, s[0].w * a.lr);
    if (a.accumulate) add4(r, j.dst[e]);
    j.dst[e] = r;
  }
}

// Sum over the 128-column blocks b = b0, b0 + step, ... < b_end of row i of the parts that the
// tail wrote past slot 0 (tiles past the whole ones; their part count read once per block, the
// slots' loads issued together).
__device__ __forceinline__ float ds_tail_slots(const float* __restrict__ part, int64_t m, int64_t nb, int64_t i,
                                               int64_t b0, int64_t step, const ReduceArgs& a, int64_t b_end = -1) {
  if (b_end < 0) b_end = nb;
  float acc = 0.0f;
  for (int64_t b = b0; b < b_end; b += step) {
    const int64_t tile = i / 128 + a.ni * (b * 128 / a.bn);
    if (tile < a.sched.full_tiles) continue;
    const int segs = __ldg(a.tile_segs + tile);
    for (int sp = 1; sp < segs; sp += 2) {
      float v[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int p = 2 * (sp + q / 2) + (q & 1);
        v[q] = sp + q / 2 < segs ? __ldg(part + (static_cast<int64_t>(p) * m + i) * nb + b) : 0.0f;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) acc += v[q];
    }
  }
  return acc;
}

// ds[i] (per channel): one warp per row; lane l sums blocks l, l + 32, ... of every
// part, then a fixed shuffle tree adds the lanes.
__device__ __forceinline__ void reduce_ds_row(const float* __restrict__ part, int nparts, int64_t m, int64_t nb,
                                              int accumulate, float* __restrict__ ds, int64_t blk,
                                              const ReduceArgs& a) {
  const int64_t i = (blk * kThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (i >= m) return;
  float acc = 0.0f;
  // parts p = 2 sp + h (slot sp, column half h); with a tail: slot 0 of every block here, the
  // written further slots of the tail's tiles below
  const int dense = a.sched.tail ? 2 : nparts;
  for (int p = 0; p < dense; ++p) {
    const float* row = part + (static_cast<int64_t>(p) * m + i) * nb;
    for (int64_t b = lane; b < nb; b += 32) acc += row[b];
  }
  if (a.sched.tail) acc += ds_tail_slots(part, m, nb, i, lane, 32, a);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (lane == 0) ds[i] = accumulate ? ds[i] + acc : acc;
}

// ds[i][g] (per group): one thread per (row, group), sequential over its blocks.
__device__ __forceinline__ void reduce_ds_group(const float* __restrict__ part, int nparts, int64_t m, int64_t nb,
                                                int ngroups, int blocks_per_group, int accumulate,
                                                float* __restrict__ ds, int64_t blk, const ReduceArgs& a) {
  const int64_t e = blk * kThreads + threadIdx.x;
  if (e >= m * ngroups) return;
  const int64_t i = e / ngroups;
  const int g = static_cast<int>(e % ngroups);
  float acc = 0.0f;
  // parts p = 2 sp + h as in reduce_ds_row
  const int dense = a.sched.tail ? 2 : nparts;
  for (int p = 0; p < dense; ++p) {
    const float* row = part + (static_cast<int64_t>(p) * m + i) * nb;
    for (int b = g * blocks_per_group; b < (g + 1) * blocks_per_group; ++b) acc += row[b];
  }
  if (a.sched.tail)
    acc += ds_tail_slots(part, m, nb, i, static_cast<int64_t>(g) * blocks_per_group, 1, a,
                         static_cast<int64_t>(g + 1) * blocks_per_group);
  ds[e] = accumulate ? ds[e] + acc : acc;
}

__global__ void __launch_bounds__(kThreads) reduce_grads_kernel(RedJob ja, RedJob jb, int64_t nblk_a, int64_t nblk_b,
                                                                ReduceArgs a, int64_t nb, int ngroups) {
  __shared__ float4 sm[kRedSlices][32];
  const int64_t blk = blockIdx.x;
  if (blk < nblk_a) {
    reduce_parts_block(ja, blk, a, sm);
  } else if (blk < nblk_a + nblk_b) {
    reduce_parts_block(jb, blk - nblk_a, a, sm);
  } else if (a.group_size == 0) {
    reduce_ds_row(a.ds_part, a.nS, a.m, nb, a.accumulate, a.ds, blk - nblk_a - nblk_b, a);
  } else {
    reduce_ds_group(a.ds_part, a.nS, a.m, nb, ngroups, a.group_size / 128, a.accumulate, a.ds,
                    blk - nblk_a - nblk_b, a);
  }
}

}  // namespace

cudaError_t launch_range_minmax(const float* W0, int64_t m, int64_t k, int group_size, int bits, float* s0,
                                float* z0, cudaStream_t stream) {
  const int ngroups = group_size ? static_cast<int>(k / group_size) : 1;
  const int seg = group_size ? group_size : static_cast<int>(k);
  const unsigned grid = static_cast<unsigned>(m * ngroups);
  if (z0 == nullptr) {
    range_minmax_kernel<<<grid, kThreads, 0, stream>>>(W0, k, seg, ngroups,
                                                       static_cast<float>((1 << (bits - 1)) - 1), s0);
  } else {
    range_minmax_asym_kernel<<<grid, kThreads, 0, stream>>>(W0, k, seg, ngroups, bits, s0, z0);
  }
  return cudaGetLastError();
}

cudaError_t launch_range_lp(const float* W0, int64_t m, int64_t k, int group_size, int bits, float p_norm, int n_cand,
                            float* s0, cudaStream_t stream) {
  const int ngroups = group_size ? static_cast<int>(k / group_size) : 1;
  const int seg = group_size ? group_size : static_cast<int>(k);
  const size_t smem = static_cast<size_t>(seg) * 4;
  if (n_cand < 1 || n_cand > kThreads || smem > 200 * 1024) return cudaErrorInvalidValue;
  if (smem > 48 * 1024) {
    // the largest row or group any call may need (200 KB), set once per device
    static bool configured[kMaxDevices] = {};
    const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(range_lp_kernel), 200 * 1024, configured);
    if (e != cudaSuccess) return e;
  }
  range_lp_kernel<<<static_cast<unsigned>(m * ngroups), kThreads, smem, stream>>>(W0, k, seg, ngroups, bits, p_norm,
                                                                                 n_cand, s0);
  return cudaGetLastError();
}

cudaError_t launch_downcast(const float* W0, const float* s0, const float* z0, int64_t m, int64_t k, int group_size,
                            int bits, int fmt, void* phi0, cudaStream_t stream) {
  const int ngroups = group_size ? static_cast<int>(k / group_size) : 1;
  const int n = -(1 << (bits - 1)), p = (1 << (bits - 1)) - 1;
  if (fmt_float(fmt)) {
    if (z0 != nullptr) return cudaErrorInvalidValue;
    const int64_t n4 = m * k / 4;
    const unsigned grid = blocks_for(n4, kThreads);
    const float4* w4 = reinterpret_cast<const float4*>(W0);
    auto kernel = fmt == FMT_BF16   ? downcast_float_kernel<FMT_BF16>
                  : fmt == FMT_F16  ? downcast_float_kernel<FMT_F16>
                  : fmt == FMT_E4M3 ? downcast_float_kernel<FMT_E4M3>
                                    : downcast_float_kernel<FMT_E5M2>;
    kernel<<<grid, kThreads, 0, stream>>>(w4, s0, k, group_size, ngroups, phi0, n4);
  } else if (fmt == FMT_Q8) {
    const int64_t n4 = m * k / 4;
    downcast_qfixed_kernel<<<blocks_for(n4, kThreads), kThreads, 0, stream>>>(
        reinterpret_cast<const float4*>(W0), s0, z0, k, group_size, ngroups, static_cast<float>(n),
        static_cast<float>(p), static_cast<float>(1 << (8 - bits)), static_cast<char4*>(phi0), n4);
  } else {
    const int64_t n8 = m * k / 8;
    downcast_packed_kernel<<<blocks_for(n8, kThreads), kThreads, 0, stream>>>(
        reinterpret_cast<const float4*>(W0), s0, z0, k, group_size, ngroups, n, p, static_cast<uint32_t*>(phi0),
        n8);
  }
  return cudaGetLastError();
}

cudaError_t launch_merge(const void* phi0, const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r,
                         int fmt, int u_bf16, const QuantParams& q, int8_t* wz, cudaStream_t stream) {
  if ((k % 4) != 0 || r > 256) return cudaErrorInvalidValue;
  const int b_aligned = (reinterpret_cast<uintptr_t>(B) & 7) == 0;
  dim3 grid(static_cast<unsigned>((k + kMergeCols - 1) / kMergeCols), static_cast<unsigned>((m + kMergeRows - 1) / kMergeRows));
  merge_kernel<<<grid, kMergeThreads, 0, stream>>>(phi0, A, B, m, k, r, fmt, u_bf16, b_aligned, q, wz);
  return cudaGetLastError();
}

cudaError_t launch_act_quant(const uint16_t* X, int64_t T, int64_t k, const float* s_x, uint16_t* codes,
                             uint32_t* mask, cudaStream_t stream) {
  if ((k % 8) != 0 || (reinterpret_cast<uintptr_t>(X) & 15) != 0 || (reinterpret_cast<uintptr_t>(codes) & 15) != 0)
    return cudaErrorInvalidValue;
  const int64_t k8 = k / 8;
  dim3 grid(static_cast<unsigned>((k8 + 7) / 8), static_cast<unsigned>((T + kAqTokens - 1) / kAqTokens));
  act_quant_kernel<<<grid, 32 * kAqWarps, 0, stream>>>(reinterpret_cast<const uint4*>(X), T, k8, s_x,
                                                       reinterpret_cast<uint4*>(codes), mask, (T + 31) / 32);
  return cudaGetLastError();
}

cudaError_t launch_act_quant_token(const uint16_t* X, int64_t T, int64_t k, uint16_t* x_hat, cudaStream_t stream) {
  if ((k % 8) != 0 || (reinterpret_cast<uintptr_t>(X) & 15) != 0 || (reinterpret_cast<uintptr_t>(x_hat) & 15) != 0)
    return cudaErrorInvalidValue;
  const int64_t k8 = k / 8;
  if (k8 <= 256 * kAtLoads) {
    int tpt_log2 = 5;
    while ((static_cast<int64_t>(1) << tpt_log2) * kAtLoads < k8) ++tpt_log2;   // 32 .. 256 threads per token
    const int64_t per_block = 256 >> tpt_log2;
    act_quant_token_kernel<<<static_cast<unsigned>((T + per_block - 1) / per_block), 256, 0, stream>>>(
        reinterpret_cast<const uint4*>(X), T, k8, tpt_log2, reinterpret_cast<uint4*>(x_hat));
  } else {
    act_quant_token_wide_kernel<<<blocks_for(T * 32, kThreads), kThreads, 0, stream>>>(
        reinterpret_cast<const uint4*>(X), T, k8, reinterpret_cast<uint4*>(x_hat));
  }
  return cudaGetLastError();
}

cudaError_t launch_adapter_layouts(const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r, int r16,
                                   uint16_t* A_pad, uint16_t* Bt_pad, uint16_t* At, uint16_t* B_pad,
                                   cudaStream_t stream) {
  if ((m % 8) != 0 || (k % 8) != 0) return cudaErrorInvalidValue;
  const int b_aligned = (reinterpret_cast<uintptr_t>(B) & 15) == 0;
  const int64_t total = (A_pad ? m * 8 : 0) + (Bt_pad ? k * 8 : 0) + (At ? static_cast<int64_t>(r16) * (m / 8) : 0) +
                        (B_pad ? static_cast<int64_t>(r16) * (k / 8) : 0);
  if (total == 0) return cudaSuccess;
  const int64_t want = blocks_for(total, kThreads);
  const unsigned grid = static_cast<unsigned>(want < 4096 ? want : 4096);
  adapter_layouts_kernel<<<grid, kThreads, 0, stream>>>(A, B, m, k, r, r16, reinterpret_cast<uint4*>(A_pad),
                                                        reinterpret_cast<uint4*>(Bt_pad), reinterpret_cast<uint4*>(At),
                                                        reinterpret_cast<uint4*>(B_pad), b_aligned);
  return cudaGetLastError();
}

cudaError_t launch_bwd_prep(const uint16_t* A, const uint16_t* B, int64_t m, int64_t k, int r, int r16,
                            uint16_t* A_pad, uint16_t* Bt_pad, uint16_t* At, uint16_t* B_pad, const void* phi0,
                            int fmt, void* phi_t, cudaStream_t stream, int clip_bits) {
  if ((m % 128) != 0 || (k % 128) != 0) return cudaErrorInvalidValue;
  const LayoutJob lj{A, B, m, k, r, r16, reinterpret_cast<uint4*>(A_pad), reinterpret_cast<uint4*>(Bt_pad),
                     reinterpret_cast<uint4*>(At), reinterpret_cast<uint4*>(B_pad),
                     (reinterpret_cast<uintptr_t>(B) & 15) == 0};
  const int64_t total = (A_pad ? m * 8 : 0) + (Bt_pad ? k * 8 : 0) + (At ? static_cast<int64_t>(r16) * (m / 8) : 0) +
                        (B_pad ? static_cast<int64_t>(r16) * (k / 8) : 0);
  const int64_t want = blocks_for(total, 256);
  const int64_t n_layout = want < 4096 ? want : 4096;
  const int64_t tile = fmt_16bit(fmt) ? 64 : 128;
  TransposeJob tj{phi0, phi_t, m, k, fmt, k / tile, 0, 0u, 0u};
  if (clip_bits > 0) {
    if (fmt != FMT_Q8 || clip_bits > 7) return cudaErrorInvalidValue;
    const uint32_t lo = static_cast<uint8_t>(-(1 << (clip_bits - 1))), hi = static_cast<uint8_t>((1 << (clip_bits - 1)) - 1);
    tj.clip = 1;
    tj.clip_lo = lo * 0x01010101u;
    tj.clip_hi = hi * 0x01010101u;
  }
  const int64_t blocks = n_layout + (k / tile) * (m / tile);
  bwd_prep_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(lj, n_layout, tj);
  return cudaGetLastError();
}

__global__ void __launch_bounds__(kThreads) dx_scales_kernel(const float* __restrict__ s, const float* __restrict__ z,
                                                             int64_t m, int groups, int s_ld, uint16_t* __restrict__ s_out,
                                                             uint16_t* __restrict__ z_out) {
  const int64_t n = m * groups;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t g = e / m, i = e % m;
    const int64_t src = s_ld ? i * s_ld + g : i;
    s_out[e] = static_cast<uint16_t>(pack_rn_bf16x2(s[src], 0.0f) & 0xffffu);
    if (z_out) z_out[e] = static_cast<uint16_t>(pack_rn_bf16x2(z[src], 0.0f) & 0xffffu);
  }
}

cudaError_t launch_dx_scales(const float* s, const float* z, int64_t m, int groups, int s_ld, uint16_t* s_out,
                             uint16_t* z_out, cudaStream_t stream) {
  const int64_t n = m * groups;
  const int grid = blocks_for(n, kThreads);
  dx_scales_kernel<<<grid < 1024 ? grid : 1024, kThreads, 0, stream>>>(s, z, m, groups, s_ld, s_out, z_out);
  return cudaGetLastError();
}

cudaError_t launch_reduce(const ReduceArgs& a, cudaStream_t stream) {
  const int64_t nA4 = a.m * a.r / 4, nB4 = static_cast<int64_t>(a.r) * a.k / 4;   // m, k are multiples of 128
  const RedJob ja{reinterpret_cast<const float4*>(a.dA_part), a.nA, nA4, reinterpret_cast<float4*>(a.dA), 0, a.r};
  const RedJob jb{reinterpret_cast<const float4*>(a.dB_part), a.nB, nB4, reinterpret_cast<float4*>(a.dB), 1, a.k};
  const int64_t nblk_a = (nA4 + 31) / 32, nblk_b = (nB4 + 31) / 32;
  const int64_t nb = a.k / 128;
  const int ngroups = a.group_size ? static_cast<int>(a.k / a.group_size) : 1;
  const int64_t nblk_s = a.group_size == 0 ? blocks_for(a.m * 32, kThreads) : blocks_for(a.m * ngroups, kThreads);
  reduce_grads_kernel<<<static_cast<unsigned>(nblk_a + nblk_b + nblk_s), kThreads, 0, stream>>>(ja, jb, nblk_a, nblk_b,
                                                                                               a, nb, ngroups);
  return cudaGetLastError();
}

}  // namespace lrqat
