"""GPU parity of the fused LR-QAT forward and backward against the oracle.

Sizes span several tiles in every dimension and leave ragged tails (token
counts that are not multiples of the 448-token forward tile or the 32-token dW
stage).  Float outputs are compared by relative Frobenius error (Y, dX: 1e-2;
dA, dB, ds: 2e-2); the integer codes the fused producers build are extracted
exactly with identity inputs and compared bit for bit, except near-ties.
"""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import DeviceLayer, bits_to_f32, near_bf16_boundary, oracle_layer, phi_host, to_dev, torch

pytestmark = pytest.mark.gpu

TOL_ACT = 1e-2
TOL_GRAD = 2e-2


def spec_of(name, m, k, r, bits=4, group=0, phi=WL.PHI_QFIXED, act=0, alpha=None, a_std=1 / 64, b_std=1e-3,
            outliers=1e-3, asym=False, shift=0.0, per_token=False, ub=False):
    return WL.LayerSpec(name, m, k, r, float(r if alpha is None else alpha), bits, group, phi, act,
                        outlier_frac=outliers, a_std=a_std, b_std=b_std, asym=asym, w_row_shift=shift,
                        act_per_token=per_token, u_bf16=ub)


def oracle_base(data, OL):
    """The oracle's own range setting and downcast: (s0, z0 or None, Phi0)."""
    if data.spec.asym:
        s0, z0 = O.minmax_range_asym(data.W0, OL)
        return s0, z0, O.downcast(data.W0, s0, OL, z0)
    s0 = O.minmax_scale(data.W0, OL)
    return s0, None, O.downcast(data.W0, s0, OL)


CASES = [
    # id, spec, T
    ("q44_pc_multi_tile", spec_of("a", 384, 512, 32), 1000),
    ("q44_pc_alpha1", spec_of("b", 256, 256, 8, alpha=1.0, a_std=0.3, b_std=0.3), 448),
    ("q35_pc_r64", spec_of("c", 128, 384, 64, bits=3, a_std=0.1, b_std=0.1), 97),
    ("int3_packed", spec_of("d", 256, 512, 32, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.2, b_std=0.2), 513),
    ("int4_packed_r4", spec_of("e", 128, 256, 4, bits=4, phi=WL.PHI_INT_PACKED, a_std=0.3, b_std=0.3), 64),
    ("q44_g128_a8", spec_of("f", 256, 384, 16, group=128, act=8, a_std=0.2, b_std=0.2), 300),
    ("q44_g256", spec_of("g", 128, 512, 32, group=256, a_std=0.2, b_std=0.2), 256),
    ("q26_clip_heavy", spec_of("h", 128, 256, 16, bits=2, a_std=1.0, b_std=1.0), 200),
    ("tokens_1", spec_of("i", 128, 128, 1), 1),
    ("q44_pc_r40", spec_of("j", 256, 256, 40, a_std=0.2, b_std=0.2), 130),
    # asymmetric weights with frozen zero offsets (the INT2 runs of the paper)
    ("int2_asym_q26_pc", spec_of("k", 256, 512, 32, bits=2, asym=True, shift=0.03, a_std=0.2, b_std=0.2), 333),
    ("int2_asym_packed_g128", spec_of("l", 128, 512, 16, bits=2, group=128, phi=WL.PHI_INT_PACKED, asym=True,
                                      shift=0.03, a_std=0.3, b_std=0.3), 200),
    ("q35_asym_g128_a8", spec_of("o", 256, 384, 32, bits=3, group=128, act=8, asym=True, shift=0.02,
                                 a_std=0.2, b_std=0.2), 150),
    # per-token dynamic int8 activations (the paper's weight-activation default)
    ("q44_pc_a8_token", spec_of("p", 256, 512, 32, act=8, per_token=True, a_std=0.2, b_std=0.2), 301),
    ("int3_packed_g128_a8_token", spec_of("q", 128, 384, 16, bits=3, group=128, phi=WL.PHI_INT_PACKED, act=8,
                                          per_token=True, a_std=0.3, b_std=0.3), 97),
    # floating-point bases (the cast choices of phi, Sec. 3)
    ("bf16_pc", spec_of("r", 256, 512, 32, phi=WL.PHI_BF16, a_std=0.2, b_std=0.2), 300),
    ("fp16_g128_w3", spec_of("s", 128, 384, 16, bits=3, group=128, phi=WL.PHI_FP16, a_std=0.2, b_std=0.2), 130),
    ("fp8_e4m3_pc_a8_token", spec_of("t", 256, 256, 16, phi=WL.PHI_FP8_E4M3, act=8, per_token=True, a_std=0.2,
                                     b_std=0.2), 200),
    ("fp8_e5m2_w2_clip", spec_of("u", 128, 512, 32, bits=2, phi=WL.PHI_FP8_E5M2, a_std=1.0, b_std=1.0), 97),
    ("bf16_w8_g128", spec_of("v", 128, 256, 8, bits=8, group=128, phi=WL.PHI_BF16, a_std=0.3, b_std=0.3), 64),
    # pre-round value in bf16 (the bf16 reading of the computation)
    ("q44_pc_ubf16", spec_of("w", 256, 512, 32, ub=True, a_std=0.2, b_std=0.2), 300),
    ("bf16_g128_ubf16_alpha1", spec_of("x", 128, 384, 16, group=128, phi=WL.PHI_BF16, alpha=1.0, ub=True,
                                       a_std=0.3, b_std=0.3), 130),
    ("int3_packed_ubf16_a8", spec_of("y", 128, 256, 16, bits=3, phi=WL.PHI_INT_PACKED, act=8, ub=True, a_std=0.3,
                                     b_std=0.3), 97),
    # ranks above 64: the codes pass writes round(u) once per call, the GEMMs read it as their
    # base and dW runs its adapter contractions in rounds of 64 ranks
    ("q44_pc_r96", spec_of("lr1", 384, 512, 96, a_std=0.1, b_std=0.1), 700),
    ("q44_pc_r128_ubf16", spec_of("lr2", 256, 512, 128, ub=True, a_std=0.1, b_std=0.1), 300),
    ("q44_pc_r256", spec_of("lr3", 256, 640, 256, a_std=0.1, b_std=0.1), 1000),
    ("int3_packed_r100", spec_of("lr4", 256, 512, 100, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.1, b_std=0.1), 513),
    ("q44_g128_a8_r200", spec_of("lr5", 256, 384, 200, group=128, act=8, a_std=0.1, b_std=0.1), 300),
    ("int2_asym_r72", spec_of("lr6", 256, 512, 72, bits=2, asym=True, shift=0.03, a_std=0.1, b_std=0.1), 333),
    ("bf16_pc_a8_token_r160", spec_of("lr7", 256, 256, 160, phi=WL.PHI_BF16, act=8, per_token=True, a_std=0.1,
                                      b_std=0.1), 200),
    ("fp8_e4m3_w2_r256_clip", spec_of("lr8", 128, 512, 256, bits=2, phi=WL.PHI_FP8_E4M3, a_std=0.2, b_std=0.2), 97),
]


def _run(spec, T, seed=0, s_scale=1.0, sx_factor=1.0, zero_B=False):
    t = torch()
    data = WL.make_layer(spec, T, seed=seed, zero_B=zero_B)
    dl = DeviceLayer(data, s_scale)
    X, dY = to_dev(data.X_bits), to_dev(data.dY_bits)
    s_x_host = None
    s_x = None
    if spec.act_bits == 8 and not spec.act_per_token:
        s_x_host = np.float32(np.float32(np.abs(data.X).max()) / np.float32(127.0) * np.float32(sx_factor))
        s_x = t.tensor([s_x_host], dtype=t.float32, device="cuda")
    L = dl.layer
    Y = t.empty((T, spec.m), dtype=t.int16, device="cuda")
    ws = t.empty(max(LQ.fwd_workspace_bytes(L, T), 16), dtype=t.uint8, device="cuda")
    LQ.linear_fwd(L, T, X, dl.phi0, dl.s, dl.A, dl.B, s_x, Y, ws)
    dX = t.empty((T, spec.k), dtype=t.int16, device="cuda")
    dA = t.empty((spec.m, spec.r), dtype=t.float32, device="cuda")
    dB = t.empty((spec.r, spec.k), dtype=t.float32, device="cuda")
    ds = t.empty_like(dl.s)
    wsb = t.empty(LQ.bwd_workspace_bytes(L, T), dtype=t.uint8, device="cuda")
    LQ.linear_bwd(L, T, dY, X, dl.phi0, dl.s, dl.A, dl.B, s_x, dX, dA, dB, ds, False, wsb)
    LQ.get_device_status()
    # oracle side: its own range setting and downcast from the same W0
    OL = oracle_layer(spec)
    s0, z0, phi0 = oracle_base(data, OL)
    if spec.asym:   # the device's zero offsets equal the oracle's exactly
        np.testing.assert_array_equal(dl.z.cpu().numpy().reshape(z0.shape), z0)
    np.testing.assert_array_equal(phi_host(dl.phi0, spec), phi0)   # and so does the stored base
    s = (s0 * np.float32(s_scale)).astype(np.float32)
    Y_ref = O.linear_fwd(data.X, phi0, s, data.A, data.B, OL, s_x_host, z0)
    g = O.linear_bwd(data.dY, data.X, phi0, s, data.A, data.B, OL, s_x_host, z0)
    got = dict(Y=bits_to_f32(Y), dX=bits_to_f32(dX), dA=dA.cpu().numpy(), dB=dB.cpu().numpy(),
               ds=ds.cpu().numpy().reshape(g["ds"].shape))
    ref = dict(Y=Y_ref, dX=g["dX"], dA=g["dA"], dB=g["dB"], ds=g["ds"])
    return got, ref, g


def with_paths(cases):
    """Each case of rank up to 64 on both sources of the GEMMs' low-rank term (the tile each
    stage computes, and the codes one pass per call writes); ranks above 64 always take the
    codes."""
    out = []
    for c in cases:
        for path in (("tile", "codes") if c[1].r <= 64 else ("auto",)):
            out.append(pytest.param(*c, path, id=f"{c[0]}-{path}"))
    return out


@pytest.mark.parametrize("cid,spec,T,path", with_paths(CASES))
def test_fwd_bwd_parity(cid, spec, T, path, lowrank_path):
    lowrank_path(path)
    got, ref, g = _run(spec, T, seed=1, s_scale=1.05)
    errs = {k: O.rel_fro(got[k], ref[k]) for k in got}
    assert errs["Y"] <= TOL_ACT and errs["dX"] <= TOL_ACT, errs
    assert errs["dA"] <= TOL_GRAD and errs["dB"] <= TOL_GRAD and errs["ds"] <= TOL_GRAD, errs
    if cid == "q26_clip_heavy":
        assert g["fq"]["M"].mean() < 0.9    # the STE clip mask matters in this case


def test_activation_clip_mask_in_dx():
    """A small activation scale clips part of X; dX must vanish there (STE mask)."""
    spec = spec_of("m", 128, 256, 16, group=128, act=8, a_std=0.2, b_std=0.2)
    got, ref, _ = _run(spec, 160, seed=4, sx_factor=0.25)
    assert (ref["dX"] == 0).mean() > 0.01
    for k in ("Y", "dX"):
        assert O.rel_fro(got[k], ref[k]) <= TOL_ACT, k
    for k in ("dA", "dB", "ds"):
        assert O.rel_fro(got[k], ref[k]) <= TOL_GRAD, k


def test_gradient_accumulation():
    """accumulate = 1 adds to dA, dB, ds; dX is overwritten."""
    t = torch()
    spec = spec_of("acc", 128, 256, 8, a_std=0.2, b_std=0.2)
    data = WL.make_layer(spec, 96, seed=9)
    dl = DeviceLayer(data)
    X, dY = to_dev(data.X_bits), to_dev(data.dY_bits)
    L = dl.layer
    ws = t.empty(LQ.bwd_workspace_bytes(L, 96), dtype=t.uint8, device="cuda")
    outs = []
    for acc in (False, True):
        dX = t.empty((96, 256), dtype=t.int16, device="cuda")
        dA = t.zeros((128, 8), dtype=t.float32, device="cuda") if not acc else outs[0][1].clone()
        dB = t.zeros((8, 256), dtype=t.float32, device="cuda") if not acc else outs[0][2].clone()
        ds = t.zeros((128,), dtype=t.float32, device="cuda") if not acc else outs[0][3].clone()
        LQ.linear_bwd(L, 96, dY, X, dl.phi0, dl.s, dl.A, dl.B, None, dX, dA, dB, ds, acc, ws)
        outs.append((dX, dA, dB, ds))
    LQ.get_device_status()
    for i in (1, 2, 3):
        np.testing.assert_allclose(outs[1][i].cpu().numpy(), 2 * outs[0][i].cpu().numpy(), rtol=1e-6, atol=1e-6)
    np.testing.assert_array_equal(outs[1][0].cpu().numpy(), outs[0][0].cpu().numpy())


CODE_CASES = [
    ("q44_pc", spec_of("c1", 256, 256, 32, a_std=0.1, b_std=0.1)),
    ("q35_pc", spec_of("c2", 128, 384, 16, bits=3, a_std=0.2, b_std=0.2)),
    ("int3_packed", spec_of("c3", 128, 256, 8, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.3, b_std=0.3)),
    ("q44_g128", spec_of("c4", 128, 256, 16, group=128, a_std=0.1, b_std=0.1)),
    ("int2_asym_q26", spec_of("c5", 128, 256, 16, bits=2, asym=True, shift=0.03, a_std=0.2, b_std=0.2)),
    ("int2_asym_packed_g128", spec_of("c6", 128, 256, 8, bits=2, group=128, phi=WL.PHI_INT_PACKED, asym=True,
                                      shift=0.03, a_std=0.3, b_std=0.3)),
    ("bf16_pc", spec_of("c7", 256, 256, 32, phi=WL.PHI_BF16, a_std=0.1, b_std=0.1)),
    ("fp16_g128", spec_of("c8", 128, 256, 16, group=128, phi=WL.PHI_FP16, a_std=0.1, b_std=0.1)),
    ("fp8_e4m3_w3", spec_of("c9", 128, 384, 16, bits=3, phi=WL.PHI_FP8_E4M3, a_std=0.2, b_std=0.2)),
    ("fp8_e5m2", spec_of("c10", 128, 256, 8, phi=WL.PHI_FP8_E5M2, a_std=0.3, b_std=0.3)),
    ("q44_pc_ubf16", spec_of("c11", 256, 256, 32, ub=True, a_std=0.3, b_std=0.3)),
    ("fp8_e4m3_ubf16_alpha1", spec_of("c12", 128, 384, 16, phi=WL.PHI_FP8_E4M3, alpha=1.0, ub=True, a_std=0.5,
                                      b_std=0.5)),
    ("q44_pc_r96", spec_of("c13", 256, 256, 96, a_std=0.1, b_std=0.1)),
    ("int3_packed_r100", spec_of("c14", 128, 256, 100, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.1, b_std=0.1)),
    ("int2_asym_g128_r256", spec_of("c15", 128, 256, 256, bits=2, group=128, asym=True, shift=0.03, a_std=0.1,
                                    b_std=0.1)),
    ("bf16_pc_r256_ubf16", spec_of("c16", 128, 256, 256, phi=WL.PHI_BF16, ub=True, a_std=0.1, b_std=0.1)),
]


@pytest.mark.parametrize("cid,spec,path", [pytest.param(c[0], c[1], p, id=f"{c[0]}-{p}") for c in CODE_CASES
                                           for p in (("tile", "codes") if c[1].r <= 64 else ("auto",))])
@pytest.mark.parametrize("zero_B", [False, True], ids=["lowrank", "ties"])
def test_fused_codes_bit_exact(cid, spec, path, zero_B, lowrank_path):
    lowrank_path(path)
    check_codes_bit_exact(cid, spec, zero_B)


def check_codes_bit_exact(cid, spec, zero_B):
    """With s = 1 and X = I (T = k) the forward returns Y = C^T exactly; with
    dY = I (T = m) the dX kernel returns its own codes C (C - z with zero offsets).
    Both must equal the oracle's codes except at near-ties; B = 0 makes every
    Q-fixed half-integer an exact tie, which both sides must round half to even."""
    t = torch()
    data = WL.make_layer(spec, 1, seed=5, with_activations=False, zero_B=zero_B)
    dl = DeviceLayer(data)
    dl.s = t.ones_like(dl.s)
    L = dl.layer
    m, k = spec.m, spec.k
    eye_k = WL.bf16_bits(np.eye(k, dtype=np.float32))
    eye_m = WL.bf16_bits(np.eye(m, dtype=np.float32))
    Y = t.empty((k, m), dtype=t.int16, device="cuda")
    ws = t.empty(max(LQ.fwd_workspace_bytes(L, k), 16), dtype=t.uint8, device="cuda")
    LQ.linear_fwd(L, k, to_dev(eye_k), dl.phi0, dl.s, dl.A, dl.B, None, Y, ws)
    T = m
    dX = t.empty((T, k), dtype=t.int16, device="cuda")
    dA = t.empty((m, spec.r), dtype=t.float32, device="cuda")
    dB = t.empty((spec.r, k), dtype=t.float32, device="cuda")
    ds = t.empty_like(dl.s)
    Xz = t.zeros((T, k), dtype=t.int16, device="cuda")
    wsb = t.empty(LQ.bwd_workspace_bytes(L, T), dtype=t.uint8, device="cuda")
    LQ.linear_bwd(L, T, to_dev(eye_m), Xz, dl.phi0, dl.s, dl.A, dl.B, None, dX, dA, dB, ds, False, wsb)
    LQ.get_device_status()
    OL = oracle_layer(spec)
    _, z0, phi0 = oracle_base(data, OL)
    ones = np.ones((m, k // spec.group_size) if spec.group_size else (m,))
    fq = O.fake_quant_weight(phi0, ones, data.A, data.B, OL, z0)
    exempt = O.near_tie(fq["u"]) if not zero_B else np.zeros_like(fq["c"], dtype=bool)
    if spec.u_bf16:   # u is a bf16 value: only the bf16 rounding of A B can differ
        exempt = near_bf16_boundary(data.A, data.B) if not zero_B else np.zeros_like(fq["c"], dtype=bool)
    c_fwd = bits_to_f32(Y).T
    c_dx = bits_to_f32(dX)
    for name, c in (("fwd", c_fwd), ("dX", c_dx)):
        bad = (c != fq["cz"]) & ~exempt
        assert bad.sum() == 0, f"{name}: {bad.sum()} code mismatches (near-ties exempt: {exempt.sum()})"
    if zero_B and spec.phi_format in (WL.PHI_QFIXED, WL.PHI_BF16, WL.PHI_FP16, WL.PHI_FP8_E4M3):
        assert (np.abs(fq["u"] - np.floor(fq["u"]) - 0.5) == 0).sum() > 0   # exact ties were exercised


def test_bf16_pre_round_moves_codes():
    """The two readings of u differ on this layer (so the bf16 cases above test something):
    the device codes follow the reading the layer asks for."""
    t = torch()
    spec = spec_of("ub", 128, 256, 8, a_std=0.05, b_std=0.05)
    data = WL.make_layer(spec, 1, seed=6, with_activations=False)
    codes = {}
    for ub in (False, True):
        sp = spec_of("ub", 128, 256, 8, a_std=0.05, b_std=0.05, ub=ub)
        dl = DeviceLayer(WL.LayerData(sp, data.W0, data.A_bits, data.B_bits))
        wz = t.empty((128, 256), dtype=t.int8, device="cuda")
        LQ.merge(dl.layer, dl.phi0, dl.A, dl.B, wz)
        LQ.get_device_status()
        codes[ub] = wz.cpu().numpy()
        OL = oracle_layer(sp)
        ref = O.merge(O.downcast(data.W0, O.minmax_scale(data.W0, OL), OL), data.A, data.B, OL)
        exempt = near_bf16_boundary(data.A, data.B) if ub else O.near_tie(
            O.preround(O.downcast(data.W0, O.minmax_scale(data.W0, OL), OL), data.A, data.B, OL))
        assert ((codes[ub] != ref) & ~exempt).sum() == 0
    assert (codes[False] != codes[True]).mean() > 0.001


@pytest.mark.parametrize("r", [8, 32, 40, 256])
def test_direct_and_padded_factor_paths_agree(r):
    """The forward reads A and B straight from the caller's arrays when they are 16-byte
    aligned (r a multiple of 8), else through padded copies; both fill the same shared
    tiles, so Y is bit-identical.  Factors shifted by one element force the padded path."""
    t = torch()
    spec = spec_of("dp", 256, 384, r, a_std=0.2, b_std=0.2)
    T = 300
    data = WL.make_layer(spec, T, seed=8)
    dl = DeviceLayer(data)
    X = to_dev(data.X_bits)
    L = dl.layer
    ws = t.empty(max(LQ.fwd_workspace_bytes(L, T), 16), dtype=t.uint8, device="cuda")
    outs = []
    for shift in (0, 1):
        A = t.empty(dl.A.numel() + 8, dtype=t.int16, device="cuda")[shift:shift + dl.A.numel()].view(dl.A.shape)
        B = t.empty(dl.B.numel() + 8, dtype=t.int16, device="cuda")[shift:shift + dl.B.numel()].view(dl.B.shape)
        A.copy_(dl.A)
        B.copy_(dl.B)
        Y = t.empty((T, spec.m), dtype=t.int16, device="cuda")
        LQ.linear_fwd(L, T, X, dl.phi0, dl.s, A, B, None, Y, ws)
        outs.append(Y.cpu().numpy())
    LQ.get_device_status()
    np.testing.assert_array_equal(outs[0], outs[1])


QUANTIZED_CASES = [
    # id, spec, T, activation scale factor (< 1 clips part of X)
    ("a8_tensor_g128_clip", spec_of("qa", 256, 384, 16, group=128, act=8, a_std=0.2, b_std=0.2), 300, 0.25),
    ("a8_token", spec_of("qb", 256, 512, 32, act=8, per_token=True, a_std=0.2, b_std=0.2), 301, 1.0),
    ("a8_tensor_packed_ubf16", spec_of("qc", 128, 256, 16, bits=3, phi=WL.PHI_INT_PACKED, act=8, ub=True,
                                       a_std=0.3, b_std=0.3), 97, 1.0),
]


@pytest.mark.parametrize("cid,spec,T,sx_factor", QUANTIZED_CASES, ids=[c[0] for c in QUANTIZED_CASES])
def test_quantized_activation_entry_points_bit_identical(cid, spec, T, sx_factor):
    """lrqat_act_quant once, then lrqat_linear_fwd_quantized / lrqat_linear_bwd_quantized on its
    codes (and clip mask): every output equals that of the entry points that quantize X
    themselves, bit for bit."""
    t = torch()
    data = WL.make_layer(spec, T, seed=9)
    dl = DeviceLayer(data)
    X, dY = to_dev(data.X_bits), to_dev(data.dY_bits)
    s_x = None
    if not spec.act_per_token:
        sx = np.float32(np.float32(np.abs(data.X).max()) / np.float32(127.0) * np.float32(sx_factor))
        s_x = t.tensor([sx], dtype=t.float32, device="cuda")
    L = dl.layer
    ws = t.empty(max(LQ.fwd_workspace_bytes(L, T), 16), dtype=t.uint8, device="cuda")
    wsb = t.empty(LQ.bwd_workspace_bytes(L, T), dtype=t.uint8, device="cuda")

    def outputs():
        return dict(Y=t.empty((T, spec.m), dtype=t.int16, device="cuda"),
                    dX=t.empty((T, spec.k), dtype=t.int16, device="cuda"),
                    dA=t.empty((spec.m, spec.r), dtype=t.float32, device="cuda"),
                    dB=t.empty((spec.r, spec.k), dtype=t.float32, device="cuda"), ds=t.empty_like(dl.s))

    a, b = outputs(), outputs()
    LQ.linear_fwd(L, T, X, dl.phi0, dl.s, dl.A, dl.B, s_x, a["Y"], ws)
    LQ.linear_bwd(L, T, dY, X, dl.phi0, dl.s, dl.A, dl.B, s_x, a["dX"], a["dA"], a["dB"], a["ds"], False, wsb)
    Xq = t.empty((T, spec.k), dtype=t.int16, device="cuda")
    mask = None if spec.act_per_token else t.empty((spec.k, (T + 31) // 32), dtype=t.int32, device="cuda")
    LQ.act_quant(L, T, X, s_x, Xq, mask)
    LQ.linear_fwd_quantized(L, T, Xq, dl.phi0, dl.s, dl.A, dl.B, s_x, b["Y"], ws)
    LQ.linear_bwd_quantized(L, T, dY, Xq, mask, dl.phi0, dl.s, dl.A, dl.B, s_x, b["dX"], b["dA"], b["dB"], b["ds"],
                            False, wsb)
    LQ.get_device_status()
    for key in a:
        assert t.equal(a[key], b[key]), key
    if sx_factor < 1.0:
        assert (bits_to_f32(b["dX"]) == 0).mean() > 0.01   # the clip mask was applied


# Ragged token counts; every tile is a tail tile (cut into token parts) except in the last case,
# which has a full wave of whole tiles (160 tiles) before its tail.
TAIL_CASES = [
    ("q44_pc", spec_of("a", 384, 512, 32), 1000),
    ("int3_packed", spec_of("d", 256, 512, 32, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.2, b_std=0.2), 1500),
    ("q44_g128_a8", spec_of("f", 256, 384, 16, group=128, act=8, a_std=0.2, b_std=0.2), 1700),
    ("int2_asym_q26", spec_of("k", 256, 512, 32, bits=2, asym=True, shift=0.03, a_std=0.2, b_std=0.2), 1300),
    ("a8_token", spec_of("p", 256, 512, 32, act=8, per_token=True, a_std=0.2, b_std=0.2), 1301),
    ("bf16_pc", spec_of("r", 256, 512, 32, phi=WL.PHI_BF16, a_std=0.2, b_std=0.2), 1250),
    ("whole_wave_then_tail", spec_of("z", 2048, 2560, 16, a_std=0.2, b_std=0.2), 650),
    ("q44_pc_r256", spec_of("lt", 256, 512, 256, a_std=0.1, b_std=0.1), 1000),
]


@pytest.mark.parametrize("cid,spec,T", TAIL_CASES, ids=[c[0] for c in TAIL_CASES])
def test_fwd_bwd_parity_tail_dw(cid, spec, T, dw_schedule):
    """The dW work with a tail (whole tiles for the full waves, then the remaining tiles cut
    into up to 8 equal token parts, one per CTA, each reduced as its own partial slot), forced
    on shapes whose cost model may pick equal splits: ragged token tails inside parts, tiles
    with different part counts, and slots that no part writes."""
    dw_schedule("tail")
    got, ref, _ = _run(spec, T, seed=2, s_scale=1.05)
    errs = {k: O.rel_fro(got[k], ref[k]) for k in got}
    assert errs["Y"] <= TOL_ACT and errs["dX"] <= TOL_ACT, errs
    assert errs["dA"] <= TOL_GRAD and errs["dB"] <= TOL_GRAD and errs["ds"] <= TOL_GRAD, errs


def test_dw_schedules_agree(dw_schedule):
    """Equal token splits and the tail schedule give the same Y and dX bit for bit and the same gradients
    up to rounding: ds up to fp32 summation order; dA and dB also up to the bf16 rounding of
    dU, which the epilogue applies per token range (about 2^-9 relative)."""
    spec = spec_of("sk", 256, 512, 32, group=128, a_std=0.2, b_std=0.2)
    outs = {}
    for sched in ("split", "tail"):
        dw_schedule(sched)
        outs[sched], _, _ = _run(spec, 1555, seed=3)
    for key in ("Y", "dX"):
        np.testing.assert_array_equal(outs["split"][key], outs["tail"][key])
    assert O.rel_fro(outs["tail"]["ds"], outs["split"]["ds"]) <= 1e-5
    for key in ("dA", "dB"):
        assert O.rel_fro(outs["tail"][key], outs["split"][key]) <= 1e-2, key


MERGE_RANK_CASES = [
    # tensor-core merge reading A and B directly (rank a multiple of 8), and the CUDA-core merge
    # (rank 100; and rank 96 with the factors shifted off 16-byte alignment), both in rank blocks
    ("q44_r256_tc", spec_of("mr1", 256, 384, 256, a_std=0.1, b_std=0.1), 0),
    ("int3_packed_r96_tc", spec_of("mr2", 128, 512, 96, bits=3, phi=WL.PHI_INT_PACKED, a_std=0.3, b_std=0.3), 0),
    ("q35_r100_cuda_cores", spec_of("mr3", 256, 256, 100, bits=3, a_std=0.2, b_std=0.2), 0),
    ("fp8_r96_shifted", spec_of("mr4", 128, 256, 96, phi=WL.PHI_FP8_E4M3, a_std=0.2, b_std=0.2), 1),
]


@pytest.mark.parametrize("cid,spec,shift", MERGE_RANK_CASES, ids=[c[0] for c in MERGE_RANK_CASES])
def test_merge_large_ranks(cid, spec, shift):
    """lrqat_merge for ranks above 64: every code equals the oracle's merge outside near-ties."""
    t = torch()
    data = WL.make_layer(spec, 1, seed=12, with_activations=False)
    dl = DeviceLayer(data)
    A = t.empty(dl.A.numel() + 8, dtype=t.int16, device="cuda")[shift:shift + dl.A.numel()].view(dl.A.shape)
    B = t.empty(dl.B.numel() + 8, dtype=t.int16, device="cuda")[shift:shift + dl.B.numel()].view(dl.B.shape)
    A.copy_(dl.A)
    B.copy_(dl.B)
    wz = t.empty((spec.m, spec.k), dtype=t.int8, device="cuda")
    LQ.merge(dl.layer, dl.phi0, A, B, wz)
    LQ.get_device_status()
    OL = oracle_layer(spec)
    _, _, phi0 = oracle_base(data, OL)
    ref = O.merge(phi0, data.A, data.B, OL)
    exempt = O.near_tie(O.preround(phi0, data.A, data.B, OL))
    assert ((wz.cpu().numpy() != ref) & ~exempt).sum() == 0
    # the factors are drawn large enough (|A B| ~ 0.5 code steps or more) that the low-rank term moves codes
    assert (ref != O.merge(phi0, data.A, np.zeros_like(data.B), OL)).mean() > 0.01


# The forward and dX GEMMs on CTA pairs (256 weight rows across two SMs) and on one SM: the
# cases whose produced operand has a multiple of 256 rows (m for the forward, k for dX) run on
# pairs when that variant is selected; both variants must match the oracle, give the same
# integer codes, and agree with each other up to fp32 summation order.
PAIR_CASES = [c for c in CASES if c[1].m % 256 == 0 or c[1].k % 256 == 0] + [
    ("q44_pc_pair_tail", spec_of("pt", 512, 768, 32, a_std=0.2, b_std=0.2), 1111),
    ("q44_g128_pair_r16", spec_of("pg", 768, 512, 16, group=128, a_std=0.2, b_std=0.2), 385),
]


@pytest.mark.parametrize("cid,spec,T,path", with_paths(PAIR_CASES))
def test_fwd_bwd_parity_gemm_variants(cid, spec, T, path, gemm_variant, lowrank_path):
    lowrank_path(path)
    outs = {}
    for variant in ("pair", "single"):
        gemm_variant(variant)
        got, ref, _ = _run(spec, T, seed=1, s_scale=1.05)
        errs = {k: O.rel_fro(got[k], ref[k]) for k in got}
        assert errs["Y"] <= TOL_ACT and errs["dX"] <= TOL_ACT, (variant, errs)
        assert errs["dA"] <= TOL_GRAD and errs["dB"] <= TOL_GRAD and errs["ds"] <= TOL_GRAD, (variant, errs)
        outs[variant] = got
    for key in ("Y", "dX"):
        assert O.rel_fro(outs["pair"][key], outs["single"][key]) <= 4e-3, key


@pytest.mark.parametrize("cid,spec", [c for c in CODE_CASES if c[1].m % 256 == 0 and c[1].k % 256 == 0],
                         ids=[c[0] for c in CODE_CASES if c[1].m % 256 == 0 and c[1].k % 256 == 0])
def test_fused_codes_bit_exact_pair_gemm(cid, spec, gemm_variant, lowrank_path):
    """The integer codes the pair kernel's producers build, through the identity inputs of
    check_codes_bit_exact, with exact ties (B = 0) and with the low-rank term, from the
    in-stage tile and from the codes pass."""
    gemm_variant("pair")
    for path in (("tile", "codes") if spec.r <= 64 else ("auto",)):
        lowrank_path(path)
        for zero_B in (False, True):
            check_codes_bit_exact(cid, spec, zero_B)
