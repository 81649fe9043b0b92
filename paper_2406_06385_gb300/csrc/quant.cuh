// Device-side arithmetic of the LR-QAT quantizer (Eq. 7 and Eq. 8 of the paper),
// written for throughput inside GEMM producer stages.
//
// With f fractional bits of the stored base (f = 8 - b for Qb.(8-b), 0 for INT-b)
// and v the stored integer (Phi0 itself, or the unpacked nibble):
//   u_f = v + 2^f (alpha/r) L            (= 2^f u, one fp32 FMA: scaling by 2^f is exact)
//   t   = u_f + 1.5 * 2^(23+f)           (fp32 add: rounds u_f to a multiple of 2^f,
//                                          ties to even, i.e. round-half-even of u)
//   t   = clamp(t, magic + 2^f n, magic + 2^f p)
//   c   = t * 2^-f - 1.5 * 2^23          (exact: the integer code clip(round(u), n, p))
// Integer inputs are turned into floats with the 2^23 exponent trick (a byte
// permute into 0x4B0000xx and one subtraction) instead of a conversion
// instruction.
#pragma once

#include <cstdint>

namespace lrqat {

// Storage formats of Phi0 (the values of lrqat_phi_format).
enum PhiFmt : int { FMT_Q8 = 0, FMT_I4 = 1, FMT_BF16 = 2, FMT_F16 = 3, FMT_E4M3 = 4, FMT_E5M2 = 5 };
__host__ __device__ constexpr bool fmt_float(int f) { return f >= FMT_BF16; }
__host__ __device__ constexpr bool fmt_16bit(int f) { return f == FMT_BF16 || f == FMT_F16; }

struct QuantParams {
  float lr_scale;   // 2^f * alpha / r
  float magic;      // 1.5 * 2^(23 + f)
  float lo;         // magic + 2^f * n
  float hi;         // magic + 2^f * p
  float inv2f;      // 2^-f
  float magic_c;    // 1.5 * 2^23
  uint32_t n_bf16x2;  // bf16 bits of n in both halves
  uint32_t p_bf16x2;  // bf16 bits of p in both halves
};

// Builds the constants above on the host.
inline QuantParams make_quant_params(int bits, int frac_bits, float alpha, int r) {
  QuantParams q;
  const double two_f = static_cast<double>(1 << frac_bits);
  const double n = -static_cast<double>(1 << (bits - 1));
  const double p = static_cast<double>((1 << (bits - 1)) - 1);
  q.lr_scale = static_cast<float>(two_f * static_cast<double>(alpha) / static_cast<double>(r));
  q.magic = static_cast<float>(1.5 * 8388608.0 * two_f);
  q.lo = static_cast<float>(1.5 * 8388608.0 * two_f + two_f * n);
  q.hi = static_cast<float>(1.5 * 8388608.0 * two_f + two_f * p);
  q.inv2f = static_cast<float>(1.0 / two_f);
  q.magic_c = 12582912.0f;   // 1.5 * 2^23
  const float nf = static_cast<float>(n), pf = static_cast<float>(p);
  uint32_t nb, pb;
  static_assert(sizeof(float) == sizeof(uint32_t), "float is 32-bit");
  __builtin_memcpy(&nb, &nf, 4);
  __builtin_memcpy(&pb, &pf, 4);
  q.n_bf16x2 = (nb >> 16) * 0x10001u;   // small integers are exact in bf16 (top 16 bits)
  q.p_bf16x2 = (pb >> 16) * 0x10001u;
  return q;
}

// Offsets that turn the exponent-trick floats of the decoders below into the
// stored integer: 2^23 + 128 for int8 bytes, 2^23 + 8 for nibbles.
constexpr float kDecodeOffsetI8 = 8388736.0f;
constexpr float kDecodeOffsetI4 = 8388616.0f;

// 4 signed bytes -> 4 floats 2^23 + (v + 128), exact (subtract kDecodeOffsetI8 for v).
__device__ __forceinline__ void decode_i8x4_raw(uint32_t w, float* f) {
  const uint32_t x = w ^ 0x80808080u;
  f[0] = __uint_as_float(__byte_perm(x, 0x4B000000u, 0x7540u));
  f[1] = __uint_as_float(__byte_perm(x, 0x4B000000u, 0x7541u));
  f[2] = __uint_as_float(__byte_perm(x, 0x4B000000u, 0x7542u));
  f[3] = __uint_as_float(__byte_perm(x, 0x4B000000u, 0x7543u));
}

// 8 signed nibbles (low nibble of byte b = element 2b) -> 8 floats 2^23 + (v + 8), exact.
__device__ __forceinline__ void decode_i4x8_raw(uint32_t w, float* f) {
  const uint32_t x = w ^ 0x88888888u;
  const uint32_t lo = x & 0x0F0F0F0Fu;
  const uint32_t hi = (x >> 4) & 0x0F0F0F0Fu;
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    f[2 * b] = __uint_as_float(__byte_perm(lo, 0x4B000000u, 0x7540u + b));
    f[2 * b + 1] = __uint_as_float(__byte_perm(hi, 0x4B000000u, 0x7540u + b));
  }
}

// Floating-point patterns -> fp32 without conversion instructions.  The pattern sits
// at the top of a 32-bit word; an arithmetic shift right by (8 - exponent bits) lines
// its exponent and mantissa fields up with fp32's and keeps the sign at bit 31, the
// mask clears the sign copies in between, and the result is the value times
// 2^(bias - 127): kFloatRebias<FMT> = 2^(127 - bias) restores it with one exact
// multiply (subnormal patterns become fp32 subnormals, which the multiply scales
// exactly; the library is built without flush-to-zero).  BF16 is the top half of fp32
// and needs nothing.  The non-finite patterns are never stored (casts saturate).
template <int FMT> struct FloatBits;
template <> struct FloatBits<FMT_E4M3> { static constexpr int kShift = 4; static constexpr uint32_t kMask = 0x87F00000u; };
template <> struct FloatBits<FMT_E5M2> { static constexpr int kShift = 3; static constexpr uint32_t kMask = 0x8FE00000u; };
template <> struct FloatBits<FMT_F16> { static constexpr int kShift = 3; static constexpr uint32_t kMask = 0x8FFFE000u; };
template <int FMT>
constexpr float kFloatRebias = FMT == FMT_E4M3 ? 1.329227995784916e36f    // 2^120
                               : FMT == FMT_BF16 ? 1.0f
                                                 : 5.192296858534828e33f;  // 2^112 (E5M2, F16)

template <int FMT>
__device__ __forceinline__ float float_bits_top(uint32_t top) {
  return __uint_as_float(static_cast<uint32_t>(static_cast<int32_t>(top) >> FloatBits<FMT>::kShift) &
                         FloatBits<FMT>::kMask);
}

// 4 FP8 patterns (byte b = element b) -> 4 floats, value * 2^(bias - 127).
template <int FMT>
__device__ __forceinline__ void decode_fp8x4_raw(uint32_t w, float* f) {
  f[0] = float_bits_top<FMT>(__byte_perm(w, 0u, 0x0444u));
  f[1] = float_bits_top<FMT>(__byte_perm(w, 0u, 0x1444u));
  f[2] = float_bits_top<FMT>(__byte_perm(w, 0u, 0x2444u));
  f[3] = float_bits_top<FMT>(__byte_perm(w, 0u, 0x3444u));
}

// 2 sixteen-bit patterns (low half = element 0) -> 2 floats (F16: value * 2^-112).
template <int FMT>
__device__ __forceinline__ void decode_16x2_raw(uint32_t w, float* f) {
  if (FMT == FMT_BF16) {
    f[0] = __uint_as_float(w << 16);
    f[1] = __uint_as_float(w & 0xFFFF0000u);
  } else {
    f[0] = float_bits_top<FMT_F16>(w << 16);
    f[1] = float_bits_top<FMT_F16>(w & 0xFFFF0000u);
  }
}

// 16 consecutive stored values of a row -> the stored values v of Eq. 8's
// u_f = v + 2^f (alpha/r) L, from the raw words (I4: 2 words, 8-bit formats: 4,
// 16-bit formats: 8).
template <int FMT>
__device__ __forceinline__ void decode16(const uint32_t* w, float* v) {
  if constexpr (FMT == FMT_I4) {
    decode_i4x8_raw(w[0], v);
    decode_i4x8_raw(w[1], v + 8);
  } else if constexpr (FMT == FMT_Q8) {
#pragma unroll
    for (int i = 0; i < 4; ++i) decode_i8x4_raw(w[i], v + 4 * i);
  } else if constexpr (fmt_16bit(FMT)) {
#pragma unroll
    for (int i = 0; i < 8; ++i) decode_16x2_raw<FMT>(w[i], v + 2 * i);
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) decode_fp8x4_raw<FMT>(w[i], v + 4 * i);
  }
  if constexpr (FMT == FMT_BF16) return;
  const float a = FMT == FMT_I4 ? 1.0f : FMT == FMT_Q8 ? 1.0f : kFloatRebias<FMT>;
  const float b = FMT == FMT_I4 ? -kDecodeOffsetI4 : FMT == FMT_Q8 ? -kDecodeOffsetI8 : 0.0f;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    float2 d;
    if (fmt_float(FMT)) d = __fmul2_rn(make_float2(v[2 * e], v[2 * e + 1]), make_float2(a, a));
    else d = __fadd2_rn(make_float2(v[2 * e], v[2 * e + 1]), make_float2(b, b));
    v[2 * e] = d.x;
    v[2 * e + 1] = d.y;
  }
}

// Exact integer codes of two elements as bf16x2, clipped to [n, p].  The
// unclipped codes are exact in fp32; bf16 keeps them exactly up to |c| <= 256 and
// truncation of larger ones keeps them beyond the clip limits, so clipping in bf16
// after packing is exact.
__device__ __forceinline__ uint32_t codes_bf16x2(float2 t, const QuantParams& q) {
  const float2 c = __ffma2_rn(t, make_float2(q.inv2f, q.inv2f), make_float2(-q.magic_c, -q.magic_c));
  uint32_t w = __byte_perm(__float_as_uint(c.x), __float_as_uint(c.y), 0x7632u);
  asm("max.bf16x2 %0, %0, %1;" : "+r"(w) : "r"(q.n_bf16x2));
  asm("min.bf16x2 %0, %0, %1;" : "+r"(w) : "r"(q.p_bf16x2));
  return w;
}

// 16 clipped codes stored offset-binary (byte = c + 128) -> their exact floats.
__device__ __forceinline__ void decode_ob16(const uint32_t* w, float* v) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
#pragma unroll
    for (int b = 0; b < 4; ++b) v[4 * i + b] = __uint_as_float(__byte_perm(w[i], 0x4B000000u, 0x7540u + b));
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const float2 d = __fadd2_rn(make_float2(v[2 * e], v[2 * e + 1]), make_float2(-kDecodeOffsetI8, -kDecodeOffsetI8));
    v[2 * e] = d.x;
    v[2 * e + 1] = d.y;
  }
}

// Four clipped codes stored as bytes c + 64 (|c| <= 64) -> two bf16x2 words: the byte becomes
// the mantissa of bf16(128 + byte) = 0x43 : byte, and one exact bf16x2 subtraction of 192
// leaves c.  w01 holds codes 0 and 1, w23 codes 2 and 3.
__device__ __forceinline__ void decode_b64_bf16x4(uint32_t w, uint32_t& w01, uint32_t& w23);

// Two exact small integers -> bf16x2 (the top halves of their floats).
__device__ __forceinline__ uint32_t pack_int_bf16x2(float c0, float c1) {
  return __byte_perm(__float_as_uint(c0), __float_as_uint(c1), 0x7632u);
}

// The same for two stored integer codes (the codes base: already rounded, 0 fraction bits):
// their floats are exact, so their top halves are their bf16 values.
__device__ __forceinline__ uint32_t int_codes_bf16x2(float c0, float c1, const QuantParams& q) {
  uint32_t w = __byte_perm(__float_as_uint(c0), __float_as_uint(c1), 0x7632u);
  asm("max.bf16x2 %0, %0, %1;" : "+r"(w) : "r"(q.n_bf16x2));
  asm("min.bf16x2 %0, %0, %1;" : "+r"(w) : "r"(q.p_bf16x2));
  return w;
}

// t = round-half-even(u_f / 2^f) in the magic domain, unclipped.
__device__ __forceinline__ float magic_round(float L, float v, const QuantParams& q) {
  const float u = __fmaf_rn(L, q.lr_scale, v);
  return __fadd_rn(u, q.magic);
}

// Integer code c = clip(round(u), n, p) as an exact float.
__device__ __forceinline__ float code_from_magic(float t, const QuantParams& q) {
  const float tc = fminf(fmaxf(t, q.lo), q.hi);
  return __fmaf_rn(tc, q.inv2f, -q.magic_c);
}

__device__ __forceinline__ float lrqat_code(float L, float v, const QuantParams& q) {
  return code_from_magic(magic_round(L, v, q), q);
}

// Two floats -> packed bf16x2 with round-to-nearest-even.
__device__ __forceinline__ uint32_t pack_rn_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Stores 16 consecutive tokens (tok0 ..) of this lane's output row, one fp32 value per token in
// v, into out [T, ld] as bf16.  Lanes (2j, 2j + 1) hold the two rows of a 4-byte word: the even
// lane writes both rows of the even tokens, the odd lane those of the odd tokens.  All eight
// shuffles are issued before any store, and one warp-uniform test covers the 16 tokens unless
// they straddle T (a shuffle-select-store chain per element with a per-element bounds test took
// ~2.3x as long in the GEMM epilogues).
__device__ __forceinline__ void store_row_pairs_bf16(const float (&v)[16], bool odd, uint16_t* out, int64_t ld,
                                                     int row, int tok0, int T) {
  float oth[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) oth[e] = __shfl_xor_sync(0xffffffffu, odd ? v[2 * e] : v[2 * e + 1], 1);
  uint32_t pk[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) pk[e] = odd ? pack_rn_bf16x2(oth[e], v[2 * e + 1]) : pack_rn_bf16x2(v[2 * e], oth[e]);
  const int t0 = tok0 + (odd ? 1 : 0);
  uint32_t* dst = reinterpret_cast<uint32_t*>(out + static_cast<int64_t>(t0) * ld + (row & ~1));
  if (tok0 + 16 <= T) {
#pragma unroll
    for (int e = 0; e < 8; ++e) dst[e * ld] = pk[e];   // two tokens = ld 4-byte words
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (t0 + 2 * e < T) dst[e * ld] = pk[e];
  }
}

// Pre-round value in bf16 (the bf16 reading of Sec. 3's computation) for two
// elements, in the units of u_f: u_f = bf16(v + bf16(lr_f bf16(L))) with lr_f =
// 2^f alpha / r a power of two, so the product is exact and one bf16 fma rounds
// exactly as the definition does; v is exact in bf16 (an integer |v| <= 128, or a
// BF16, FP8 or nibble value), its fp32 low half zero.
__device__ __forceinline__ float2 u_bf16x2(float L0, float L1, float v0, float v1, uint32_t lr2) {
  const uint32_t lb = pack_rn_bf16x2(L0, L1);
  const uint32_t vb = __byte_perm(__float_as_uint(v0), __float_as_uint(v1), 0x7632u);
  uint32_t u;
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(u) : "r"(lb), "r"(lr2), "r"(vb));
  return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xFFFF0000u));
}

// Elementwise bf16x2 difference, rounded to nearest even (exact for the small
// integers it is used on).
__device__ __forceinline__ uint32_t sub_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ void decode_b64_bf16x4(uint32_t w, uint32_t& w01, uint32_t& w23) {
  w01 = sub_bf16x2(__byte_perm(w, 0x43u, 0x4140u), 0x43404340u);
  w23 = sub_bf16x2(__byte_perm(w, 0x43u, 0x4342u), 0x43404340u);
}

// Elementwise bf16x2 product, rounded to nearest even.
__device__ __forceinline__ uint32_t mul_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

__device__ __forceinline__ float bf16_to_float(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

}  // namespace lrqat
