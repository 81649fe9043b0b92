"""Seeded synthetic workloads for the LR-QAT linear layer.

This module only draws random numbers and rounds them to the storage types the
layer consumes (fp32 weights, bf16 adapters and activations).  It contains none
of the method's arithmetic: no scale estimation, no downcast, no rounding to the
quantization grid.  Both the CPU oracle and the CUDA path receive the arrays
produced here, so the two sides always see identical bytes.

Shapes follow the paper's models (LLaMA-2 7B/13B and LLaMA-3 8B linear layers,
Sec. 4 and Appendix B): attention projections d x d, MLP projections d -> d_ff
-> d.  The paper trains on SlimPajama sequences (batch 32 x 1024 tokens,
Sec. 4, Table B1); that data is not available here, so activations and output
gradients are i.i.d. normal stand-ins of the same token counts.

Random streams: numpy PCG64 seeded through ``SeedSequence(seed)``; every layer
spawns one child sequence and every tensor draws from its own grandchild, in
the fixed order W0, outlier positions, A, B, X, dY.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import List, Optional

import numpy as np

PHI_QFIXED = 0       # int8 fixed point Qb.(8-b), Eq. 7
PHI_INT_PACKED = 1   # two INT-b nibbles per byte (Sec. 3, downcasting operator)
PHI_BF16 = 2         # floating-point casts of W0 / s0 (Sec. 3), stored as bit patterns
PHI_FP16 = 3
PHI_FP8_E4M3 = 4
PHI_FP8_E5M2 = 5


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bfloat16 (round to nearest even); return raw uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> 16).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of raw bfloat16 bits to fp32."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclass(frozen=True)
class LayerSpec:
    """Shape and quantizer settings of one LR-QAT linear layer (W is m x k)."""
    name: str
    m: int                 # out features
    k: int                 # in features
    r: int                 # adapter rank
    alpha: float           # LoRA scaling numerator (alpha / r multiplies A B)
    bits: int              # weight bit-width b
    group_size: int        # 0 = per output channel, else group width along k
    phi_format: int        # one of the PHI_* storage formats above
    act_bits: int = 0      # 0 = no activation quantizer, 8 = per-tensor int8
    w_std: float = 0.02
    outlier_frac: float = 0.0
    outlier_mult: float = 10.0
    a_std: float = 0.01
    b_std: float = 0.01
    asym: bool = False     # asymmetric weights: zero offsets z (the INT2 runs of the paper)
    w_row_shift: float = 0.0   # each row of W0 shifted by U(-w_row_shift, w_row_shift)
    act_per_token: bool = False   # with act_bits 8: dynamic per-token scales (else per tensor)
    u_bf16: bool = False   # pre-round value formed in bf16 instead of fp32


@dataclass(frozen=True)
class Workload:
    """A named set of layers that one fwd+bwd step processes, all with T tokens."""
    name: str
    tokens: int
    layers: List[LayerSpec] = field(default_factory=list)
    merge: bool = False
    x_std: float = 1.0
    dy_std: float = 1.0

    def flops_fwd_bwd(self) -> float:
        """Dense GEMM FLOPs of one fwd+bwd step: 2*T*m*k for each of Y, dX and dW."""
        return float(sum(6.0 * self.tokens * l.m * l.k for l in self.layers))


def _llama_layer(name, m, k, *, bits, group_size, phi_format, act_bits=0):
    return LayerSpec(name=name, m=m, k=k, r=32, alpha=32.0, bits=bits, group_size=group_size,
                     phi_format=phi_format, act_bits=act_bits, w_std=0.02, outlier_frac=1e-3,
                     outlier_mult=10.0, a_std=1.0 / 64.0, b_std=1e-3)


def workload(name: str) -> Workload:
    """The five layer workloads the benchmark and the parity tests use.

    tiny            : 256x256, T=64, r=4, alpha=4, W4 per channel, Q4.4
    llama2_7b_attn  : 4096x4096, T=8192, r=32, W4 per channel, Q4.4
    llama2_7b_mlp   : gate/up 4096->11008, down 11008->4096, T=8192, W3 per channel, packed INT-3
    llama3_8b_mlp   : 4096->14336->4096, T=8192, W4 g128, per-tensor int8 activations, Q4.4
    llama2_13b_layer: q/k/v/o 5120^2, gate/up 5120->13824, down 13824->5120, T=16384, W4 pc, Q4.4, merge
    llama2_7b_attn_int2: 4096x4096, T=8192, r=32, W2 per channel asymmetric (frozen zero
                      offsets, the paper's INT2 setting), Q2.6
    llama2_7b_attn_w4a8: 4096x4096, T=8192, r=32, W4 per channel, Q4.4, per-token dynamic int8
                      activations (the paper's weight-activation default)
    llama2_7b_attn_r256: the 4096x4096 layer at rank 256, alpha = 256
    """
    if name == "tiny":
        return Workload(name, 64, [LayerSpec("proj", 256, 256, r=4, alpha=4.0, bits=4, group_size=0,
                                             phi_format=PHI_QFIXED, w_std=0.02, a_std=0.01, b_std=0.01)])
    if name == "llama2_7b_attn":
        return Workload(name, 8192, [_llama_layer("attn", 4096, 4096, bits=4, group_size=0,
                                                  phi_format=PHI_QFIXED)])
    if name == "llama2_7b_mlp":
        kw = dict(bits=3, group_size=0, phi_format=PHI_INT_PACKED)
        return Workload(name, 8192, [_llama_layer("gate", 11008, 4096, **kw),
                                     _llama_layer("up", 11008, 4096, **kw),
                                     _llama_layer("down", 4096, 11008, **kw)])
    if name == "llama3_8b_mlp":
        kw = dict(bits=4, group_size=128, phi_format=PHI_QFIXED, act_bits=8)
        return Workload(name, 8192, [_llama_layer("gate", 14336, 4096, **kw),
                                     _llama_layer("up", 14336, 4096, **kw),
                                     _llama_layer("down", 4096, 14336, **kw)])
    if name == "llama2_13b_layer":
        kw = dict(bits=4, group_size=0, phi_format=PHI_QFIXED)
        return Workload(name, 16384, [_llama_layer(n, 5120, 5120, **kw) for n in ("q", "k", "v", "o")]
                        + [_llama_layer("gate", 13824, 5120, **kw), _llama_layer("up", 13824, 5120, **kw),
                           _llama_layer("down", 5120, 13824, **kw)], merge=True)
    if name == "llama2_7b_attn_int2":
        spec = _llama_layer("attn", 4096, 4096, bits=2, group_size=0, phi_format=PHI_QFIXED)
        return Workload(name, 8192, [replace(spec, asym=True)])
    if name == "llama2_7b_attn_w4a8":
        spec = _llama_layer("attn", 4096, 4096, bits=4, group_size=0, phi_format=PHI_QFIXED, act_bits=8)
        return Workload(name, 8192, [replace(spec, act_per_token=True)])
    if name == "llama2_7b_attn_ubf16":
        # the bench layer with its pre-round value formed in bf16 (the bf16 reading of Sec. 3)
        spec = _llama_layer("attn", 4096, 4096, bits=4, group_size=0, phi_format=PHI_QFIXED)
        return Workload(name, 8192, [replace(spec, u_bf16=True)])
    if name == "llama2_7b_attn_r256":
        # the bench layer at the largest rank of the paper's rank ablation (Sec. 4.1, App. A)
        spec = _llama_layer("attn", 4096, 4096, bits=4, group_size=0, phi_format=PHI_QFIXED)
        return Workload(name, 8192, [replace(spec, r=256, alpha=256.0)])
    if name.startswith("llama2_7b_attn_phi_"):
        # the same 4096 x 4096 W4 per-channel layer with a floating-point base (Table 2 ablation)
        fmt = {"bf16": PHI_BF16, "fp16": PHI_FP16, "fp8": PHI_FP8_E4M3, "fp8e5m2": PHI_FP8_E5M2}[name[19:]]
        return Workload(name, 8192, [_llama_layer("attn", 4096, 4096, bits=4, group_size=0, phi_format=fmt)])
    raise KeyError(f"unknown workload {name!r}")


WORKLOADS = ("tiny", "llama2_7b_attn", "llama2_7b_mlp", "llama3_8b_mlp", "llama2_13b_layer", "llama2_7b_attn_int2",
             "llama2_7b_attn_w4a8", "llama2_7b_attn_phi_bf16", "llama2_7b_attn_phi_fp16", "llama2_7b_attn_phi_fp8",
             "llama2_7b_attn_phi_fp8e5m2", "llama2_7b_attn_ubf16", "llama2_7b_attn_r256")


@dataclass
class LayerData:
    """Host arrays of one layer.  bf16 tensors are kept both as raw bits (what the
    device receives) and as their exact fp32 values (what the oracle receives)."""
    spec: LayerSpec
    W0: np.ndarray          # fp32 [m, k]
    A_bits: np.ndarray      # uint16 [m, r]
    B_bits: np.ndarray      # uint16 [r, k]
    X_bits: Optional[np.ndarray] = None    # uint16 [T, k]
    dY_bits: Optional[np.ndarray] = None   # uint16 [T, m]

    @property
    def A(self) -> np.ndarray:
        return bf16_to_f32(self.A_bits)

    @property
    def B(self) -> np.ndarray:
        return bf16_to_f32(self.B_bits)

    @property
    def X(self) -> np.ndarray:
        return bf16_to_f32(self.X_bits)

    @property
    def dY(self) -> np.ndarray:
        return bf16_to_f32(self.dY_bits)


def make_layer(spec: LayerSpec, tokens: int, seed: int = 0, layer_index: int = 0,
               with_activations: bool = True, x_std: float = 1.0, dy_std: float = 1.0,
               zero_B: bool = False) -> LayerData:
    """Draw one layer's weights, adapters and (optionally) a batch of T tokens.

    Outliers: round(outlier_frac * m * k) positions, drawn without replacement,
    are multiplied by ``outlier_mult`` before anything else looks at W0.
    ``zero_B`` replaces B by zeros (the LoRA initialisation, Sec. 4.2), which puts
    every fixed-point half-integer of Phi0 exactly on a rounding tie.
    """
    ss = np.random.SeedSequence(seed).spawn(layer_index + 1)[layer_index]
    g_w, g_o, g_a, g_b, g_x, g_dy = [np.random.Generator(np.random.PCG64(s)) for s in ss.spawn(6)]
    m, k, r = spec.m, spec.k, spec.r
    W0 = g_w.standard_normal((m, k), dtype=np.float32) * np.float32(spec.w_std)
    n_out = int(round(spec.outlier_frac * m * k))
    if n_out > 0:
        pos = g_o.choice(m * k, size=n_out, replace=False)
        W0.reshape(-1)[pos] *= np.float32(spec.outlier_mult)
    if spec.w_row_shift > 0:
        g_s = np.random.Generator(np.random.PCG64(ss.spawn(1)[0]))
        W0 += g_s.uniform(-spec.w_row_shift, spec.w_row_shift, size=(m, 1)).astype(np.float32)
    A_bits = bf16_bits(g_a.standard_normal((m, r), dtype=np.float32) * np.float32(spec.a_std))
    if zero_B:
        B_bits = np.zeros((r, k), dtype=np.uint16)
    else:
        B_bits = bf16_bits(g_b.standard_normal((r, k), dtype=np.float32) * np.float32(spec.b_std))
    data = LayerData(spec, W0, A_bits, B_bits)
    if with_activations:
        data.X_bits = bf16_bits(g_x.standard_normal((tokens, k), dtype=np.float32) * np.float32(x_std))
        data.dY_bits = bf16_bits(g_dy.standard_normal((tokens, m), dtype=np.float32) * np.float32(dy_std))
    return data


def token_sample(n_tokens: int, n_sample: int, seed: int = 0) -> np.ndarray:
    """Sorted, distinct token indices for checks that sample rows of a large batch."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, 0x5A])))
    return np.sort(g.choice(n_tokens, size=min(n_sample, n_tokens), replace=False))
