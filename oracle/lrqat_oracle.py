"""CPU oracle for the LR-QAT linear layer (arXiv 2406.06385).

TEST INFRASTRUCTURE ONLY.  This module is the independent reference that the
CUDA path is checked against.  Only the test suite, ``__graft_entry__.smoke``
and the CPU-baseline leg of ``bench.py`` may import it; the library itself never
does.  It shares no code with the CUDA path and imports nothing from it: every
function below is written from the paper's equations, in float64 unless the
paper (or the reading stated next to the function) fixes another precision.

Notation (Sec. 3 of the paper): a linear layer y = W x with W in R^{m x k}
(m = out features, k = in features); tokens are stacked as rows, so
Y[T, m] = X[T, k] W^T.  Bit-width b gives the symmetric integer grid
[n, p] = [-2^{b-1}, 2^{b-1} - 1] (Eq. 1, Eq. 3).

  * Eq. 6 / Eq. 7   Phi0 = phi(W0 / s0): frozen downcast of the pretrained weight
  * Eq. 8           W_hat = s * clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p)
  * Eq. 4 text      gradients w.r.t. A, B, s use the straight-through estimator
                    d round(t) / dt = 1 (first introduced with Eq. 3)
  * Sec. 3 end      after training W_Z = clip(...) is the integer weight, W_hat = s W_Z

Readings where the paper is silent (all repeated in the design notes):
  R1 round(.) is round-half-to-even (IEEE round-to-nearest; what PyTorch's
     torch.round does, and the paper's implementation is PyTorch, App. B).
  R2 the pre-round value u = phi^{-1}(Phi0) + (alpha/r) A B is formed at full
     precision; integer codes are compared exactly except where the fp32
     rendering of u lies within 1e-5 of a half-integer (see ``near_tie``).
  R3 the STE clip mask is taken on the rounded value: M = 1[n <= round(u) <= p].
  R4 ds is the plain gradient sum_j G_ij c_ij (no LSQ gradient scaling).
  R5 per-channel scales are per output row; groups (g128) run along k.
  R6 the nibble order of double packing: low nibble = even column, high nibble
     = odd column, 4-bit two's complement.
  R7 s0 comes from symmetric min-max range setting: max|W0| over the row (or
     group) divided by p, in fp32; an all-zero row/group gets s0 = 1.
  R8 W0 / s0 in the downcast is one fp32 IEEE division (the result then decides
     an integer code, so both sides take it in the same precision).
  R9 activation quantizer (weight-activation runs): per-tensor symmetric int8,
     X_Z = clip(round(X / s_x), -128, 127) with X / s_x one fp32 division,
     X_hat = s_x X_Z, STE with clip mask M_x = 1[-128 <= round(X/s_x) <= 127].
  R13 asymmetric weights (the INT2 runs of Sec. 4; Eq. 1 with the zero offset z
     outside the rounding, as the end of Sec. 3 states): W_hat = s (W_Z - z) with
     W_Z = clip(round(phi^{-1}(Phi0) + (alpha/r) A B + z), n, p) and z frozen at its
     range-setting value z0 (Sec. 4).  z is an integer, so round(x) + z = round(x + z)
     and the oracle stores Phi0 = phi(W0 / s0 + z0): the frozen base already carries
     the offset and Eq. 8's clip range stays [n, p].  Range setting is asymmetric
     min-max: s0 = (max - min) / (2^b - 1) in fp32 and z0 = clip(round(n - min / s0),
     n, p) with min / s0 one fp32 division and the rest exact.  The STE mask is
     unchanged and ds = sum G (W_Z - z).
  R14 per-token activations (the default of the weight-activation runs, Sec. 4):
     dynamic absmax scale per token, s_x[t] = max_j |X[t, j]| / 127 in fp32 (1 for
     an all-zero token), X_Z = clip(round(X / s_x[t]), -128, 127) with X / s_x[t] one
     fp32 division, X_hat = s_x[t] X_Z; the scale is not differentiated (STE with
     the clip mask, as R9).
  R17 optimizer step (App. B, Table B1): AdamW with decoupled weight decay
     (Loshchilov & Hutter), (beta1, beta2) = (0.9, 0.95), bias-corrected moments,
     eps = 1e-8 (not stated; the usual default), separate learning rates for A, B
     and for s, weight decay 0 by default; before it, clipping of the global L2 norm
     of all trainable gradients to max_norm = 1.0 with coefficient
     min(1, max_norm / (norm + 1e-6)).  A and B are updated in fp32 master copies.
  R18 L^p range setting (App. B, the alternative to min-max): per row (or group)
     the scale minimising sum |w - s clip(round(w / s), n, p)|^p over the candidates
     s_j = fl32(s_minmax * j / N), j = 1..N (N = 100), w / s_j one fp32 division;
     the smallest j wins a tie.  Symmetric grids only.
  R19 floating-point downcasting operators (Sec. 3 names FP16, BF16 and FP8 as the
     simplest choices of phi): Phi0 = cast(fl32(W0 / s0)) with round-to-nearest-even
     and no clipping inside phi (the clip of Eq. 8 follows the low-rank add); FP8 is
     the OCP E4M3 (bias 7, no infinities, largest finite 448) or E5M2 (bias 15,
     largest finite 57344) format; FP16 and FP8 casts beyond the largest finite
     value saturate to it.  phi^{-1} is the exact value.  Stored as bit patterns: uint16
     for BF16/FP16, uint8 for FP8.  Symmetric grids only.
  R20 bf16 pre-round variant (the reading that R2 rejects, kept to measure it):
     u = bf16(phi^{-1}(Phi0) + bf16((alpha/r) bf16(A B))), each product and sum
     rounded to bf16 as an eager bf16 implementation would (A B from the exact sum).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, Optional

import numpy as np

PHI_QFIXED = 0
PHI_INT_PACKED = 1
PHI_BF16 = 2
PHI_FP16 = 3
PHI_FP8_E4M3 = 4
PHI_FP8_E5M2 = 5
FLOAT_PHI = (PHI_BF16, PHI_FP16, PHI_FP8_E4M3, PHI_FP8_E5M2)

NEAR_TIE_TOL = 1e-5


@dataclass(frozen=True)
class Layer:
    """Quantizer settings of one layer, as the oracle sees them."""
    m: int
    k: int
    r: int
    alpha: float
    bits: int
    group_size: int = 0          # 0 = per output channel
    phi_format: int = PHI_QFIXED
    act_bits: int = 0            # 0 or 8
    act_per_token: bool = False  # with act_bits 8: one dynamic scale per token (R14)
    u_bf16: bool = False         # pre-round value in bf16 (R20) instead of full precision (R2)


def grid(bits: int):
    """Symmetric b-bit integer grid [n, p] of Eq. 1 with z = 0."""
    return -(2 ** (bits - 1)), 2 ** (bits - 1) - 1


def frac_bits(layer: Layer) -> int:
    """Fractional bits of the stored Phi0: 8 - b for Qb.(8-b) (Eq. 7), 0 for INT-b."""
    return 8 - layer.bits if layer.phi_format == PHI_QFIXED else 0


def expand_scale(s: np.ndarray, layer: Layer) -> np.ndarray:
    """Broadcast a per-row [m] or per-group [m, k/g] scale to the full [m, k] shape (R5)."""
    s = np.asarray(s, dtype=np.float64)
    if layer.group_size == 0:
        return np.repeat(s.reshape(layer.m, 1), layer.k, axis=1)
    return np.repeat(s.reshape(layer.m, layer.k // layer.group_size), layer.group_size, axis=1)


# ----------------------------------------------------------------------------
# Range setting (App. B "PTQ initialization", min-max estimator) -- reading R7
# ----------------------------------------------------------------------------
def minmax_scale(W0: np.ndarray, layer: Layer) -> np.ndarray:
    """s0 = max|W0| / p over each output row (or each g-wide group of a row), fp32."""
    _, p = grid(layer.bits)
    W0 = np.asarray(W0, dtype=np.float32)
    if layer.group_size == 0:
        amax = np.abs(W0).max(axis=1)
    else:
        amax = np.abs(W0.reshape(layer.m, layer.k // layer.group_size, layer.group_size)).max(axis=2)
    safe = np.where(amax > 0, amax, np.float32(p)).astype(np.float32)
    return np.divide(safe, np.float32(p), dtype=np.float32)


def minmax_range_asym(W0: np.ndarray, layer: Layer):
    """Asymmetric min-max range setting (reading R13): returns (s0, z0), both float32
    and shaped like the scales; z0 holds integers in [n, p]."""
    n, p = grid(layer.bits)
    W0 = np.asarray(W0, dtype=np.float32)
    if layer.group_size == 0:
        seg = W0.reshape(layer.m, 1, layer.k)
    else:
        seg = W0.reshape(layer.m, layer.k // layer.group_size, layer.group_size)
    lo = seg.min(axis=2).astype(np.float32)
    hi = seg.max(axis=2).astype(np.float32)
    span = np.subtract(hi, lo, dtype=np.float32)
    span = np.where(span > 0, span, np.float32(2 ** layer.bits - 1)).astype(np.float32)
    s0 = np.divide(span, np.float32(2 ** layer.bits - 1), dtype=np.float32)
    q = np.divide(lo, s0, dtype=np.float32).astype(np.float64)
    z0 = np.clip(np.rint(n - q), n, p).astype(np.float32)
    if layer.group_size == 0:
        return s0.reshape(layer.m), z0.reshape(layer.m)
    return s0, z0


def expand_zero(z: Optional[np.ndarray], layer: Layer) -> np.ndarray:
    """The zero offsets broadcast to [m, k] (0 for a symmetric layer)."""
    if z is None:
        return np.zeros((layer.m, layer.k))
    return expand_scale(z, layer)


def lp_candidates(s_max: np.ndarray, n_cand: int) -> np.ndarray:
    """Candidate scales s_j = fl32(s_max * j / N), j = 1..N, as float32 [..., N] (R18)."""
    j = np.arange(1, n_cand + 1, dtype=np.float64)
    return (np.asarray(s_max, dtype=np.float64)[..., None] * j / n_cand).astype(np.float32)


def lp_loss(w: np.ndarray, s: float, bits: int, p_norm: float) -> float:
    """sum |w - s clip(round(w / s), n, p)|^p for one row or group (Eq. 1 quantizer, z = 0)."""
    n, p = grid(bits)
    w32 = np.asarray(w, dtype=np.float32)
    q = np.clip(np.rint(np.divide(w32, np.float32(s), dtype=np.float32).astype(np.float64)), n, p)
    return float(np.sum(np.abs(w32.astype(np.float64) - float(s) * q) ** p_norm))


def lp_range(W0: np.ndarray, layer: Layer, p_norm: float, n_cand: int = 100):
    """L^p range setting (R18): returns (s0 float32 shaped like the scales, chosen j - 1)."""
    s_max = minmax_scale(W0, layer)
    W0 = np.asarray(W0, dtype=np.float32)
    segs = W0.reshape(layer.m, -1, layer.group_size if layer.group_size else layer.k)
    cands = lp_candidates(s_max.reshape(layer.m, -1), n_cand)
    best = np.zeros(segs.shape[:2], dtype=np.int64)
    for i in range(segs.shape[0]):
        for g in range(segs.shape[1]):
            losses = [lp_loss(segs[i, g], cands[i, g, j], layer.bits, p_norm) for j in range(n_cand)]
            best[i, g] = int(np.argmin(losses))       # first minimum: the smallest j wins a tie
    s0 = np.take_along_axis(cands, best[..., None], axis=2)[..., 0]
    return s0.reshape(s_max.shape), best.reshape(s_max.shape)


# ----------------------------------------------------------------------------
# Downcasting operator phi and its inverse (Sec. 3, Eq. 6, Eq. 7)
# ----------------------------------------------------------------------------
def pack_nibbles(codes: np.ndarray) -> np.ndarray:
    """Double packing of INT-b values (b <= 4) into bytes, reading R6.

    Byte j of a row holds column 2j in its low nibble and column 2j+1 in its
    high nibble, each as a 4-bit two's complement number.
    """
    codes = np.asarray(codes).astype(np.int64)
    assert codes.shape[1] % 2 == 0
    assert codes.min(initial=0) >= -8 and codes.max(initial=0) <= 7
    lo = codes[:, 0::2] & 0xF          # two's complement low 4 bits
    hi = codes[:, 1::2] & 0xF
    return (lo | (hi << 4)).astype(np.uint8)


def unpack_nibbles(packed: np.ndarray) -> np.ndarray:
    """Inverse of ``pack_nibbles``: sign-extend each nibble back to an integer."""
    packed = np.asarray(packed, dtype=np.uint8).astype(np.int64)
    lo = packed & 0xF
    hi = packed >> 4
    out = np.empty((packed.shape[0], 2 * packed.shape[1]), dtype=np.int64)
    out[:, 0::2] = np.where(lo >= 8, lo - 16, lo)
    out[:, 1::2] = np.where(hi >= 8, hi - 16, hi)
    return out.astype(np.int8)


# ----------------------------------------------------------------------------
# Floating-point storage formats of phi (Sec. 3) -- reading R19
# ----------------------------------------------------------------------------
_FP8_LAYOUT = {PHI_FP8_E4M3: (4, 3, 7), PHI_FP8_E5M2: (5, 2, 15)}   # exponent bits, mantissa bits, bias


def fp8_value(code: int, fmt: int) -> float:
    """Value of one FP8 bit pattern from the format's definition (NaN for the
    non-finite patterns): sign, biased exponent e, mantissa m; e = 0 is subnormal,
    m / 2^M * 2^(1 - bias); otherwise (1 + m / 2^M) * 2^(e - bias).  E4M3 has no
    infinities and only S.1111.111 is NaN; E5M2 reserves e = 31 as IEEE does."""
    eb, mb, bias = _FP8_LAYOUT[fmt]
    sign = -1.0 if code & 0x80 else 1.0
    e = (code >> mb) & ((1 << eb) - 1)
    m = code & ((1 << mb) - 1)
    if fmt == PHI_FP8_E4M3 and e == 15 and m == 7:
        return float("nan")
    if fmt == PHI_FP8_E5M2 and e == 31:
        return float("nan")
    if e == 0:
        return sign * (m / 2.0 ** mb) * 2.0 ** (1 - bias)
    return sign * (1.0 + m / 2.0 ** mb) * 2.0 ** (e - bias)


def fp8_encode(x: np.ndarray, fmt: int) -> np.ndarray:
    """Round-to-nearest-even cast of fp32 values to FP8 bit patterns, saturating at
    the largest finite magnitude (R19).  The nearest finite magnitude is found on
    the table of all non-negative finite values (ascending with the code); on an
    exact midpoint the even code (even mantissa) wins.  The sign bit is kept, so a
    negative value that rounds to zero gives negative zero."""
    mags = np.array([fp8_value(c, fmt) for c in range(128)])
    finite = np.nonzero(np.isfinite(mags))[0]
    grid_v, grid_c = mags[finite], finite
    x = np.asarray(x)
    if x.dtype != np.float64:   # float64 inputs are rounded from their own value
        x = x.astype(np.float32)
    a = np.minimum(np.abs(x.astype(np.float64)), grid_v[-1])
    hi = np.clip(np.searchsorted(grid_v, a, side="left"), 0, len(grid_v) - 1)
    lo = np.maximum(hi - 1, 0)
    d_lo, d_hi = a - grid_v[lo], grid_v[hi] - a
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (grid_c[hi] % 2 == 0))
    code = np.where(pick_hi, grid_c[hi], grid_c[lo]).astype(np.uint8)
    return code | np.where(np.signbit(x), np.uint8(0x80), np.uint8(0))


def fp8_decode(codes: np.ndarray, fmt: int) -> np.ndarray:
    table = np.array([fp8_value(c, fmt) for c in range(256)])
    return table[np.asarray(codes, dtype=np.uint8).astype(np.int64)]


def bf16_encode(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even of fp32 values to bf16 (the upper half of the fp32 bit
    pattern), as uint16 bit patterns: add 0x7FFF plus the lowest kept bit, truncate.
    (Finite inputs only; they never come near the fp32 overflow threshold here.)"""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((b + 0x7FFF + ((b >> 16) & 1)) >> 16).astype(np.uint16)


def bf16_round(v: np.ndarray) -> np.ndarray:
    """float64 values in bf16's normal range rounded (nearest, ties to even) to the 8
    significant bits of bf16, in one step: v = m 2^e with m in [0.5, 1), keep
    rint(m 2^8) 2^(e-8)."""
    m, e = np.frexp(np.asarray(v, dtype=np.float64))
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def bf16_decode(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def float_cast(x: np.ndarray, fmt: int) -> np.ndarray:
    """phi for the floating-point formats: the stored bit patterns of x (R19)."""
    if fmt == PHI_BF16:
        return bf16_encode(x)
    if fmt == PHI_FP16:   # saturating at the largest finite fp16, 65504
        return np.clip(np.asarray(x, dtype=np.float32), -65504.0, 65504.0).astype(np.float16).view(np.uint16)
    return fp8_encode(x, fmt)


def float_value(bits: np.ndarray, fmt: int) -> np.ndarray:
    """phi^{-1} for the floating-point formats: the exact value as float64."""
    if fmt == PHI_BF16:
        return bf16_decode(bits)
    if fmt == PHI_FP16:
        return np.asarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)
    return fp8_decode(bits, fmt)


def downcast(W0: np.ndarray, s0: np.ndarray, layer: Layer, z0: Optional[np.ndarray] = None) -> np.ndarray:
    """Phi0 = phi(W0 / s0) (Eq. 6); with zero offsets phi(W0 / s0 + z0) (reading R13).

    Q-fixed (Eq. 7): INT8(round(2^{8-b} * clip(x, n, p))), stored int8 [m, k].
    INT-b (Sec. 3): clip(round(x), n, p), double-packed into uint8 [m, k/2].
    BF16 / FP16 / FP8 (R19): the rounded cast of x, as bit patterns.
    W0 / s0 is a single fp32 division per element (reading R8); adding the integer
    offset is exact.
    """
    n, p = grid(layer.bits)
    W0 = np.asarray(W0, dtype=np.float32)
    s_full = expand_scale(s0, layer).astype(np.float32)
    x32 = np.divide(W0, s_full, dtype=np.float32)
    if layer.phi_format in FLOAT_PHI:
        if z0 is not None:
            raise ValueError("floating-point phi is defined for symmetric grids only (R19)")
        return float_cast(x32, layer.phi_format)
    x = x32.astype(np.float64)
    if z0 is not None:
        x = x + expand_scale(z0, layer)
    if layer.phi_format == PHI_QFIXED:
        y = np.clip(x, n, p) * 2.0 ** (8 - layer.bits)
        return np.rint(y).astype(np.int8)
    codes = np.clip(np.rint(x), n, p).astype(np.int8)
    return pack_nibbles(codes)


def downcast_fp64_changes(W0: np.ndarray, s0: np.ndarray, layer: Layer,
                          z0: Optional[np.ndarray] = None) -> np.ndarray:
    """Mask of the elements whose stored base would change if W0 / s0 were one float64
    division instead of the fp32 IEEE division the downcast uses (reading R8): the
    value phi^{-1}(Phi0) of ``downcast`` against the same format rounded from the
    float64 quotient."""
    n, p = grid(layer.bits)
    ref = upcast(downcast(W0, s0, layer, z0), layer)
    x = np.asarray(W0, dtype=np.float32).astype(np.float64) / expand_scale(s0, layer).astype(np.float32).astype(np.float64)
    if z0 is not None:
        x = x + expand_scale(z0, layer)
    fmt = layer.phi_format
    if fmt == PHI_QFIXED:
        f = 2.0 ** (8 - layer.bits)
        alt = np.rint(np.clip(x, n, p) * f) / f
    elif fmt == PHI_INT_PACKED:
        alt = np.clip(np.rint(x), n, p)
    elif fmt == PHI_BF16:
        alt = bf16_round(x)
    elif fmt == PHI_FP16:
        alt = np.clip(x, -65504.0, 65504.0).astype(np.float16).astype(np.float64)
    else:
        alt = fp8_decode(fp8_encode(x, fmt), fmt)
    return ref != alt


def upcast(Phi0: np.ndarray, layer: Layer) -> np.ndarray:
    """phi^{-1}(Phi0) as float64: Phi0 / 2^{8-b} (Eq. 7), the unpacked INT-b value, or
    the exact value of a floating-point pattern (R19)."""
    if layer.phi_format in FLOAT_PHI:
        return float_value(Phi0, layer.phi_format)
    if layer.phi_format == PHI_QFIXED:
        return np.asarray(Phi0, dtype=np.int8).astype(np.float64) / 2.0 ** (8 - layer.bits)
    return unpack_nibbles(Phi0).astype(np.float64)


# ----------------------------------------------------------------------------
# LR-QAT weight (Eq. 8) and its integer codes
# ----------------------------------------------------------------------------
def preround(Phi0: np.ndarray, A: np.ndarray, B: np.ndarray, layer: Layer) -> np.ndarray:
    """u = phi^{-1}(Phi0) + (alpha / r) A B, the argument of round() in Eq. 8 (reading R2;
    with ``layer.u_bf16`` each step rounded to bf16, reading R20)."""
    AB = np.asarray(A, dtype=np.float64) @ np.asarray(B, dtype=np.float64)
    if layer.u_bf16:
        bf = bf16_round
        return bf(upcast(Phi0, layer) + bf((layer.alpha / layer.r) * bf(AB)))
    return upcast(Phi0, layer) + (layer.alpha / layer.r) * AB


def codes_from_u(u: np.ndarray, layer: Layer):
    """q = round(u) (R1), c = clip(q, n, p) (Eq. 8), M = 1[n <= q <= p] (R3)."""
    n, p = grid(layer.bits)
    q = np.rint(u)
    c = np.clip(q, n, p)
    M = ((q >= n) & (q <= p)).astype(np.float64)
    return q, c, M


def near_tie(u: np.ndarray, tol: float = NEAR_TIE_TOL) -> np.ndarray:
    """Elements whose fp32 pre-round value lies within ``tol`` of a half-integer.

    There the rounding decision depends on the last bits of the low-rank sum, so
    two correct implementations may pick different codes.
    """
    u32 = np.asarray(u, dtype=np.float32).astype(np.float64)
    return np.abs(u32 - (np.floor(u32) + 0.5)) <= tol


def fake_quant_weight(Phi0, s, A, B, layer: Layer, z: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
    """W_hat = s * clip(round(phi^{-1}(Phi0) + (alpha/r) A B), n, p)  (Eq. 8);
    with zero offsets W_hat = s * (clip(...) - z), the offset carried by Phi0 (R13)."""
    u = preround(Phi0, A, B, layer)
    q, c, M = codes_from_u(u, layer)
    cz = c - expand_zero(z, layer)
    return {"u": u, "q": q, "c": c, "cz": cz, "M": M, "W_hat": expand_scale(s, layer) * cz}


def merge(Phi0, A, B, layer: Layer) -> np.ndarray:
    """Integer weight W_Z = clip(round(...), n, p) that training leaves behind (Sec. 3, Eq. 8);
    with zero offsets the dequantized weight is s (W_Z - z) (Eq. 1)."""
    return codes_from_u(preround(Phi0, A, B, layer), layer)[1].astype(np.int8)


# ----------------------------------------------------------------------------
# Activation quantizer (weight-activation runs, Sec. 4 "Quantization") -- R9
# ----------------------------------------------------------------------------
def act_quant(X: np.ndarray, s_x: float):
    """Per-tensor symmetric int8 fake quantization of activations (Eq. 1, z = 0, b = 8)."""
    x = np.divide(np.asarray(X, dtype=np.float32), np.float32(s_x), dtype=np.float32)
    q = np.rint(x.astype(np.float64))
    codes = np.clip(q, -128, 127)
    mask = ((q >= -128) & (q <= 127)).astype(np.float64)
    return codes, float(np.float32(s_x)) * codes, mask


def act_scale_per_token(X: np.ndarray) -> np.ndarray:
    """Dynamic per-token absmax scales s_x[t] = max_j |X[t, j]| / 127, fp32 (R14)."""
    amax = np.abs(np.asarray(X, dtype=np.float32)).max(axis=1)
    amax = np.where(amax > 0, amax, np.float32(127.0)).astype(np.float32)
    return np.divide(amax, np.float32(127.0), dtype=np.float32)


def act_quant_per_token(X: np.ndarray):
    """Per-token int8 fake quantization (Eq. 1, z = 0, b = 8, one scale per token):
    returns (codes, X_hat, mask, s_x)."""
    s_x = act_scale_per_token(X)
    x = np.divide(np.asarray(X, dtype=np.float32), s_x[:, None], dtype=np.float32)
    q = np.rint(x.astype(np.float64))
    codes = np.clip(q, -128, 127)
    mask = ((q >= -128) & (q <= 127)).astype(np.float64)
    return codes, s_x.astype(np.float64)[:, None] * codes, mask, s_x


# ----------------------------------------------------------------------------
# Linear layer forward / backward with checkpointed W_hat (Sec. 3)
# ----------------------------------------------------------------------------
def _inputs(X, layer: Layer, s_x: Optional[float]):
    X = np.asarray(X, dtype=np.float64)
    if layer.act_bits == 8 and layer.act_per_token:
        _, Xh, Mx, _ = act_quant_per_token(X)
        return Xh, Mx
    if layer.act_bits == 8:
        assert s_x is not None
        _, Xh, Mx = act_quant(X, s_x)
        return Xh, Mx
    return X, np.ones_like(X)


def linear_fwd(X, Phi0, s, A, B, layer: Layer, s_x: Optional[float] = None,
               z: Optional[np.ndarray] = None) -> np.ndarray:
    """Y = X_hat W_hat^T with W_hat from Eq. 8; returns float64 [T, m]."""
    Xh, _ = _inputs(X, layer, s_x)
    return Xh @ fake_quant_weight(Phi0, s, A, B, layer, z)["W_hat"].T


def linear_bwd(dY, X, Phi0, s, A, B, layer: Layer, s_x: Optional[float] = None,
               z: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
    """Gradients of the LR-QAT layer for an upstream gradient dY [T, m].

    W_hat is recomputed from Phi0, A, B, s (the checkpointing of Sec. 3).  With
    G = dY^T X_hat (the gradient w.r.t. W_hat) and the STE of Eq. 3/4:
      dX = (dY W_hat) * M_x
      dU = G * s * M                    (gradient w.r.t. u, mask from R3)
      dA = (alpha/r) dU B^T,  dB = (alpha/r) A^T dU
      ds = sum over the row (or group) of G * c   (reading R4; G * (c - z), R13)
    """
    dY = np.asarray(dY, dtype=np.float64)
    Xh, Mx = _inputs(X, layer, s_x)
    fq = fake_quant_weight(Phi0, s, A, B, layer, z)
    dX = (dY @ fq["W_hat"]) * Mx
    G = dY.T @ Xh
    dU = G * expand_scale(s, layer) * fq["M"]
    scale = layer.alpha / layer.r
    dA = scale * (dU @ np.asarray(B, dtype=np.float64).T)
    dB = scale * (np.asarray(A, dtype=np.float64).T @ dU)
    Gc = G * fq["cz"]
    if layer.group_size == 0:
        ds = Gc.sum(axis=1)
    else:
        ds = Gc.reshape(layer.m, layer.k // layer.group_size, layer.group_size).sum(axis=2)
    return {"dX": dX, "dA": dA, "dB": dB, "ds": ds, "G": G, "fq": fq}


def linear_bwd_loops(dY, X, Phi0, s, A, B, layer: Layer, s_x: Optional[float] = None,
                     z: Optional[np.ndarray] = None) -> Dict[str, np.ndarray]:
    """The same gradients as ``linear_bwd``, hand-expanded into scalar loops.

    For tiny shapes only.  Each weight element is rebuilt from Eq. 8 with its
    own rank-r dot product, and each gradient is accumulated term by term with
    the chain rule through s * clip(round(.)) under the STE.
    """
    n, p = grid(layer.bits)
    T = len(dY)
    m, k, r = layer.m, layer.k, layer.r
    P = upcast(Phi0, layer)
    s_full = expand_scale(s, layer)
    z_full = expand_zero(z, layer)
    Xh, Mx = _inputs(X, layer, s_x)
    A = np.asarray(A, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    dY = np.asarray(dY, dtype=np.float64)
    scale = layer.alpha / layer.r
    dX = np.zeros((T, k))
    dA = np.zeros((m, r))
    dB = np.zeros((r, k))
    ds = np.zeros((m,) if layer.group_size == 0 else (m, k // layer.group_size))
    for i in range(m):
        for j in range(k):
            lowrank = 0.0
            for t in range(r):
                lowrank += A[i, t] * B[t, j]
            u = P[i, j] + scale * lowrank
            q = float(np.rint(u))
            c = min(max(q, n), p)
            inside = 1.0 if n <= q <= p else 0.0
            w = s_full[i, j] * (c - z_full[i, j])
            g = 0.0                              # dL/dW_hat[i, j] = sum_tok dY[tok, i] X_hat[tok, j]
            for tok in range(T):
                g += dY[tok, i] * Xh[tok, j]
                dX[tok, j] += dY[tok, i] * w * Mx[tok, j]
            du = g * s_full[i, j] * inside       # STE through round, zero outside the clip range
            for t in range(r):
                dA[i, t] += scale * du * B[t, j]
                dB[t, j] += scale * du * A[i, t]
            if layer.group_size == 0:
                ds[i] += g * (c - z_full[i, j])
            else:
                ds[i, j // layer.group_size] += g * (c - z_full[i, j])
    return {"dX": dX, "dA": dA, "dB": dB, "ds": ds}


# ----------------------------------------------------------------------------
# Optimizer step on the trainable parameters A, B, s (App. B, Table B1) -- R17
# ----------------------------------------------------------------------------
def clip_coefficient(grads, max_norm: float) -> float:
    """Global L2-norm clipping: all gradients are multiplied by this coefficient."""
    total = float(np.sqrt(sum(float(np.sum(np.asarray(g, dtype=np.float64) ** 2)) for g in grads)))
    return min(1.0, max_norm / (total + 1e-6))


def adamw_update(p, g, m, v, step: int, lr: float, beta1: float = 0.9, beta2: float = 0.95, eps: float = 1e-8,
                 weight_decay: float = 0.0):
    """One AdamW step (decoupled weight decay) for one tensor; returns (p, m, v) as float64.

    step counts from 1.  The moments are bias-corrected; the decay multiplies the
    parameter by (1 - lr * weight_decay) before the Adam update, which is the same
    as subtracting lr * weight_decay * p from it.
    """
    p = np.asarray(p, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    m = beta1 * np.asarray(m, dtype=np.float64) + (1.0 - beta1) * g
    v = beta2 * np.asarray(v, dtype=np.float64) + (1.0 - beta2) * g * g
    m_hat = m / (1.0 - beta1 ** step)
    v_hat = v / (1.0 - beta2 ** step)
    p = p * (1.0 - lr * weight_decay) - lr * m_hat / (np.sqrt(v_hat) + eps)
    return p, m, v


def rel_fro(a: np.ndarray, b: np.ndarray) -> float:
    """Relative Frobenius error ||a - b|| / ||b|| (the parity metric for float outputs)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / den) if den > 0 else float(np.linalg.norm(a - b))
