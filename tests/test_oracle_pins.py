"""Pins of the CPU oracle against facts the paper and the mathematics fix.

None of these tests compares the oracle with itself: each checks it against a
hand-worked example, a special case with a known answer, an exhaustive
enumeration, an exact finite difference, or a library autograd of a closed form.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import workloads as WL


# ---------------------------------------------------------------------------
# Hand-worked example, Eq. 7 (phi = Q4.4) and Eq. 8, b = 4, r = 1, alpha = 1: the inputs
# and every intermediate value (dyadic rationals worked out by hand) are in
# tests/golden/hand_example_q44.json.
# ---------------------------------------------------------------------------
with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_example_q44.json")) as _f:
    HAND = json.load(_f)
_HL = HAND["layer"]
HAND_LAYER = O.Layer(m=_HL["m"], k=_HL["k"], r=_HL["r"], alpha=_HL["alpha"], bits=_HL["bits"])
HAND_W0 = np.array(HAND["inputs"]["W0"], dtype=np.float32)
HAND_A = np.array(HAND["inputs"]["A"])
HAND_B = np.array(HAND["inputs"]["B"])
HAND_S = np.array(HAND["inputs"]["s"])            # trained scale, differs from s0 on purpose
HAND_X = np.array(HAND["inputs"]["X"])
HAND_DY = np.array(HAND["inputs"]["dY"])
HAND_STEP = HAND["steps"]


def test_hand_example_downcast_and_codes():
    s0 = O.minmax_scale(HAND_W0, HAND_LAYER)
    np.testing.assert_array_equal(s0, np.array(HAND_STEP["s0 = max|W0 row| / 7"], dtype=np.float32))
    phi0 = O.downcast(HAND_W0, s0, HAND_LAYER)
    np.testing.assert_array_equal(phi0, HAND_STEP["Phi0 = 16 x"])
    fq = O.fake_quant_weight(phi0, HAND_S, HAND_A, HAND_B, HAND_LAYER)
    np.testing.assert_array_equal(fq["u"], HAND_STEP["u = Phi0/16 + (alpha/r) A B"])
    np.testing.assert_array_equal(fq["q"], HAND_STEP["q = round_half_even(u)"])
    np.testing.assert_array_equal(fq["c"], HAND_STEP["c = clip(q, -8, 7)"])
    np.testing.assert_array_equal(fq["M"], HAND_STEP["M = [n <= q <= p]"])
    np.testing.assert_array_equal(fq["W_hat"], HAND_STEP["W_hat = s c"])
    np.testing.assert_array_equal(O.merge(phi0, HAND_A, HAND_B, HAND_LAYER), HAND_STEP["c = clip(q, -8, 7)"])


def test_hand_example_forward_backward():
    phi0 = np.array(HAND_STEP["Phi0 = 16 x"], dtype=np.int8)
    Y = O.linear_fwd(HAND_X, phi0, HAND_S, HAND_A, HAND_B, HAND_LAYER)
    np.testing.assert_array_equal(Y, HAND_STEP["Y = X W_hat^T"])
    g = O.linear_bwd(HAND_DY, HAND_X, phi0, HAND_S, HAND_A, HAND_B, HAND_LAYER)
    np.testing.assert_array_equal(g["dX"], HAND_STEP["dX = dY W_hat"])
    np.testing.assert_array_equal(g["G"], HAND_STEP["G = dY^T X"])
    np.testing.assert_array_equal(g["dA"], HAND_STEP["dA = (alpha/r) dU B^T"])
    np.testing.assert_array_equal(g["dB"], HAND_STEP["dB = (alpha/r) A^T dU"])
    np.testing.assert_array_equal(g["ds"], HAND_STEP["ds = sum_k G c"])


def test_hand_example_alpha_over_r_half():
    # Same weights with alpha = 0.5, r = 1: (alpha/r) A B = row 0 [0.375, 0.25, -0.125, 0.09375],
    # row 1 [-0.1875, -0.125, 0.0625, -0.046875];  u row 0 = [7.375, -3.25, 1.125, 0.40625] (no clip now),
    # u row 1 = [-7.1875, 3.625, 0.1875, 6.453125];  q = [[7, -3, 1, 0], [-7, 4, 0, 6]], M = 1 everywhere.
    # dU row 0 = 0.25 * [1, 1.5, 0, 1] = [0.25, 0.375, 0, 0.25]; dU row 1 = [-0.5, -2, 2.5, 0.75]
    # dA = 0.5 * dU B^T = [[0.421875], [-1.859375]];  dB = 0.5 * A^T dU = [[0.125, 0.34375, -0.3125, -0.03125]]
    layer = O.Layer(m=2, k=4, r=1, alpha=0.5, bits=4)
    phi0 = np.array([[112, -56, 20, 5], [-112, 60, 2, 104]], dtype=np.int8)
    fq = O.fake_quant_weight(phi0, HAND_S, HAND_A, HAND_B, layer)
    np.testing.assert_array_equal(fq["u"], [[7.375, -3.25, 1.125, 0.40625], [-7.1875, 3.625, 0.1875, 6.453125]])
    np.testing.assert_array_equal(fq["c"], [[7, -3, 1, 0], [-7, 4, 0, 6]])
    assert fq["M"].min() == 1.0
    g = O.linear_bwd(HAND_DY, HAND_X, phi0, HAND_S, HAND_A, HAND_B, layer)
    np.testing.assert_array_equal(g["dA"], [[0.421875], [-1.859375]])
    np.testing.assert_array_equal(g["dB"], [[0.125, 0.34375, -0.3125, -0.03125]])
    np.testing.assert_array_equal(g["ds"], [2.5, 0.0])


def test_hand_example_int4_packed():
    # phi = INT-4 (Sec. 3): codes clip(round(x)) = row 0 [7, -4, 1, 0], row 1 [-7, 4, 0, 6]
    # packed bytes: row 0 [0xC7, 0x01], row 1 [0x49, 0x60]
    layer = O.Layer(m=2, k=4, r=1, alpha=1.0, bits=4, phi_format=O.PHI_INT_PACKED)
    s0 = O.minmax_scale(HAND_W0, layer)
    phi0 = O.downcast(HAND_W0, s0, layer)
    np.testing.assert_array_equal(phi0, np.array([[0xC7, 0x01], [0x49, 0x60]], dtype=np.uint8))
    np.testing.assert_array_equal(O.upcast(phi0, layer), [[7, -4, 1, 0], [-7, 4, 0, 6]])
    # u row 0 = [7.75, -3.5, 0.75, 0.1875] -> q = [8, -4, 1, 0] (-3.5 ties to even -4)
    fq = O.fake_quant_weight(phi0, HAND_S, HAND_A, HAND_B, layer)
    np.testing.assert_array_equal(fq["q"][0], [8, -4, 1, 0])
    np.testing.assert_array_equal(fq["c"][0], [7, -4, 1, 0])
    np.testing.assert_array_equal(fq["M"][0], [0, 1, 1, 1])


def test_hand_example_activation_quantizer():
    # s_x = 0.5: X / s_x = [2, 4, -2, 1] ... all inside [-128, 127]
    codes, xh, mask = O.act_quant(HAND_X, 0.5)
    np.testing.assert_array_equal(codes, HAND_X * 2)
    np.testing.assert_array_equal(xh, HAND_X)
    assert mask.min() == 1.0
    # s_x = 1/64: 2 * 64 = 128 -> clipped to 127, mask 0; -1 * 64 = -64 and -2 * 64 = -128 stay;
    # 1.984375 * 64 = 127 stays; 1.9921875 * 64 = 127.5 ties to even 128 -> clipped, mask 0
    codes, xh, mask = O.act_quant(np.array([[2.0, -1.0, -2.0, 1.984375, 1.9921875]]), 1.0 / 64)
    np.testing.assert_array_equal(codes, [[127, -64, -128, 127, 127]])
    np.testing.assert_array_equal(mask, [[0, 1, 1, 1, 0]])


def test_minmax_zero_row_and_groups():
    layer = O.Layer(m=2, k=256, r=1, alpha=1.0, bits=3, group_size=128)
    W0 = np.zeros((2, 256), dtype=np.float32)
    W0[0, 5] = -1.5          # group (0, 0): max 1.5 -> 1.5 / 3 = 0.5
    W0[1, 200] = 0.75        # group (1, 1): 0.75 / 3 = 0.25
    np.testing.assert_array_equal(O.minmax_scale(W0, layer), [[0.5, 1.0], [1.0, 0.25]])


def test_near_tie_rule():
    u = np.array([0.5, 0.500005, 0.5001, -2.499995, 3.0, 1.4999])
    np.testing.assert_array_equal(O.near_tie(u), [True, True, False, True, False, False])


# ---------------------------------------------------------------------------
# Special cases with a textbook answer
# ---------------------------------------------------------------------------
def _rtn_python(x32: np.ndarray, n: int, p: int) -> np.ndarray:
    """Round-to-nearest PTQ (Eq. 1 with z = 0) via Python's built-in round (half to even)."""
    out = np.empty(x32.shape, dtype=np.int64)
    for idx in np.ndindex(x32.shape):
        out[idx] = min(max(round(float(x32[idx])), n), p)
    return out


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_int_phi_with_zero_adapter_is_rtn(bits):
    """phi = INT-b and B = 0: W_Z equals round-to-nearest quantization of W0 exactly."""
    layer = O.Layer(m=24, k=64, r=4, alpha=4.0, bits=bits, phi_format=O.PHI_INT_PACKED)
    spec = WL.LayerSpec("t", 24, 64, 4, 4.0, bits, 0, WL.PHI_INT_PACKED, outlier_frac=0.01)
    d = WL.make_layer(spec, 1, seed=3, zero_B=True, with_activations=False)
    s0 = O.minmax_scale(d.W0, layer)
    x32 = np.divide(d.W0, s0[:, None].astype(np.float32), dtype=np.float32)
    n, p = O.grid(bits)
    wz = O.merge(O.downcast(d.W0, s0, layer), d.A, d.B, layer)
    np.testing.assert_array_equal(wz, _rtn_python(x32, n, p))


@pytest.mark.parametrize("bits", [3, 4])
def test_qfixed_with_zero_adapter_is_rtn_except_double_rounding(bits):
    """phi = Qb.(8-b) and B = 0: W_Z equals RTN of W0 except where the stored value
    round(2^f x)/2^f lands exactly on a half-integer that x itself is not on
    (double rounding); that set is predicted in closed form and must match exactly."""
    layer = O.Layer(m=64, k=128, r=4, alpha=4.0, bits=bits)
    spec = WL.LayerSpec("t", 64, 128, 4, 4.0, bits, 0, WL.PHI_QFIXED, outlier_frac=0.01)
    d = WL.make_layer(spec, 1, seed=5, zero_B=True, with_activations=False)
    s0 = O.minmax_scale(d.W0, layer)
    x32 = np.divide(d.W0, s0[:, None].astype(np.float32), dtype=np.float32)
    n, p = O.grid(bits)
    f = 8 - bits
    wz = O.merge(O.downcast(d.W0, s0, layer), d.A, d.B, layer).astype(np.int64)
    rtn = _rtn_python(x32, n, p)
    stored = np.array([round(min(max(float(v), n), p) * 2 ** f) / 2 ** f for v in x32.ravel()]).reshape(x32.shape)
    on_half = (stored - np.floor(stored)) == 0.5
    predicted = on_half & (np.vectorize(lambda a, b: round(a) != min(max(round(b), n), p))(stored, x32.astype(np.float64)))
    mismatch = wz != rtn
    np.testing.assert_array_equal(mismatch, predicted)
    assert mismatch.sum() > 0   # the set is not empty on this draw


@pytest.mark.parametrize("bits", [2, 3, 4, 5, 6, 7])
def test_qfixed_grid_round_trip_exhaustive(bits):
    """Every Qb.(8-b) grid value j / 2^{8-b} survives phi^{-1}(phi(.)) exactly (Eq. 7)."""
    n, p = O.grid(bits)
    f = 8 - bits
    js = np.arange(n * 2 ** f, p * 2 ** f + 1)
    layer = O.Layer(m=1, k=len(js), r=1, alpha=1.0, bits=bits)
    v = (js / 2 ** f).astype(np.float32)[None, :]
    s0 = np.ones(1, dtype=np.float32)
    phi = O.downcast(v, s0, layer)
    np.testing.assert_array_equal(phi[0], js)
    np.testing.assert_array_equal(O.upcast(phi, layer)[0], v[0])
    np.testing.assert_array_equal(O.downcast(O.upcast(phi, layer).astype(np.float32), s0, layer), phi)
    assert phi.min() == -128 and phi.max() == p * 2 ** f


def test_nibble_packing_exhaustive():
    """All 256 bytes unpack and re-pack to themselves; all 256 nibble pairs round-trip."""
    allbytes = np.arange(256, dtype=np.uint8).reshape(1, 256)
    np.testing.assert_array_equal(O.pack_nibbles(O.unpack_nibbles(allbytes)), allbytes)
    pairs = np.array(list(itertools.product(range(-8, 8), repeat=2)), dtype=np.int64).reshape(1, -1)
    np.testing.assert_array_equal(O.unpack_nibbles(O.pack_nibbles(pairs)), pairs)
    # low nibble is the even column (reading R6)
    np.testing.assert_array_equal(O.pack_nibbles(np.array([[1, -1]])), [[0xF1]])


@pytest.mark.parametrize("phi_format,bits", [(O.PHI_QFIXED, 4), (O.PHI_QFIXED, 3), (O.PHI_INT_PACKED, 3)])
def test_code_range_with_large_adapters(phi_format, bits):
    """Codes stay on the b-bit grid whatever A B does; Phi0 stays in its storage range."""
    layer = O.Layer(m=32, k=64, r=8, alpha=8.0, bits=bits, phi_format=phi_format)
    spec = WL.LayerSpec("t", 32, 64, 8, 8.0, bits, 0, phi_format, a_std=2.0, b_std=2.0)
    d = WL.make_layer(spec, 1, seed=7, with_activations=False)
    s0 = O.minmax_scale(d.W0, layer)
    phi0 = O.downcast(d.W0, s0, layer)
    n, p = O.grid(bits)
    if phi_format == O.PHI_QFIXED:
        assert phi0.min() >= -128 and phi0.max() <= p * 2 ** (8 - bits)
    fq = O.fake_quant_weight(phi0, s0, d.A, d.B, layer)
    assert fq["c"].min() == n and fq["c"].max() == p     # large A B pushes both clip ends
    assert 0 < fq["M"].mean() < 1


@pytest.mark.parametrize("group_size", [0, 128])
def test_merge_reproduces_fake_quant_weight(group_size):
    """s * W_Z == W_hat element by element (Sec. 3: no loss when folding the adapters)."""
    layer = O.Layer(m=16, k=256, r=4, alpha=4.0, bits=4, group_size=group_size)
    spec = WL.LayerSpec("t", 16, 256, 4, 4.0, 4, group_size, WL.PHI_QFIXED, a_std=0.3, b_std=0.3)
    d = WL.make_layer(spec, 1, seed=11, with_activations=False)
    s0 = O.minmax_scale(d.W0, layer)
    phi0 = O.downcast(d.W0, s0, layer)
    s = s0 * np.float32(1.1)
    wz = O.merge(phi0, d.A, d.B, layer)
    fq = O.fake_quant_weight(phi0, s, d.A, d.B, layer)
    np.testing.assert_array_equal(O.expand_scale(s, layer) * wz, fq["W_hat"])


# ---------------------------------------------------------------------------
# Gradients: matrix form vs hand-expanded loops, finite differences, autograd
# ---------------------------------------------------------------------------
LOOP_CASES = [
    dict(m=4, k=6, r=2, bits=4, group_size=0, phi=O.PHI_QFIXED, act=0, std=0.3),
    dict(m=4, k=6, r=2, bits=3, group_size=0, phi=O.PHI_QFIXED, act=0, std=2.0),      # clip active
    dict(m=3, k=8, r=3, bits=4, group_size=0, phi=O.PHI_INT_PACKED, act=0, std=1.0),
    dict(m=2, k=256, r=2, bits=4, group_size=128, phi=O.PHI_QFIXED, act=0, std=1.0),
    dict(m=4, k=6, r=2, bits=4, group_size=0, phi=O.PHI_QFIXED, act=8, std=1.0),
    dict(m=4, k=6, r=2, bits=4, group_size=0, phi=O.PHI_BF16, act=0, std=0.3),
    dict(m=4, k=6, r=2, bits=3, group_size=0, phi=O.PHI_FP8_E4M3, act=0, std=2.0),    # clip active
    dict(m=2, k=256, r=2, bits=4, group_size=128, phi=O.PHI_FP16, act=0, std=1.0),
]


def _tiny(case, T=3, seed=13):
    layer = O.Layer(case["m"], case["k"], case["r"], float(case["r"]), case["bits"], case["group_size"],
                    case["phi"], case["act"])
    spec = WL.LayerSpec("t", case["m"], case["k"], case["r"], float(case["r"]), case["bits"],
                        case["group_size"], case["phi"], a_std=case["std"], b_std=case["std"])
    d = WL.make_layer(spec, T, seed=seed)
    s0 = O.minmax_scale(d.W0, layer)
    phi0 = O.downcast(d.W0, s0, layer)
    s = s0 * np.float32(0.9)
    s_x = float(np.abs(d.X).max()) / 200.0 if case["act"] else None   # small s_x: some clipping
    return layer, d, phi0, s, s_x


@pytest.mark.parametrize("case", LOOP_CASES)
def test_ste_gradients_match_scalar_loops(case):
    layer, d, phi0, s, s_x = _tiny(case)
    ref = O.linear_bwd_loops(d.dY, d.X, phi0, s, d.A, d.B, layer, s_x)
    got = O.linear_bwd(d.dY, d.X, phi0, s, d.A, d.B, layer, s_x)
    for name in ("dX", "dA", "dB", "ds"):
        np.testing.assert_allclose(got[name], ref[name], rtol=1e-12, atol=1e-12, err_msg=name)
    if case["std"] == 2.0:
        assert got["fq"]["M"].min() == 0.0       # the clip mask is exercised
    if case["act"]:
        assert O.act_quant(d.X, s_x)[2].min() == 0.0


def _loss(dY, X, phi0, s, A, B, layer):
    return float(np.sum(dY * O.linear_fwd(X, phi0, s, A, B, layer)))


@pytest.mark.parametrize("case", LOOP_CASES[:4] + LOOP_CASES[5:])
def test_dX_and_ds_are_exact_gradients(case):
    """Y is linear in X and in s (c does not depend on s, Eq. 5/8), so central
    differences of <dY, Y> reproduce dX and ds up to float64 rounding."""
    layer, d, phi0, s, _ = _tiny(case, T=4)
    g = O.linear_bwd(d.dY, d.X, phi0, s, d.A, d.B, layer)
    eps = 0.5
    for (t, j) in [(0, 0), (1, layer.k - 1), (3, layer.k // 2)]:
        Xp, Xm = d.X.astype(np.float64).copy(), d.X.astype(np.float64).copy()
        Xp[t, j] += eps
        Xm[t, j] -= eps
        fd = (_loss(d.dY, Xp, phi0, s, d.A, d.B, layer) - _loss(d.dY, Xm, phi0, s, d.A, d.B, layer)) / (2 * eps)
        assert abs(fd - g["dX"][t, j]) <= 1e-9 * max(1.0, abs(fd))
    s64 = s.astype(np.float64)
    for idx in [(0,) if s.ndim == 1 else (0, 0), (layer.m - 1,) if s.ndim == 1 else (layer.m - 1, 1)]:
        sp, sm = s64.copy(), s64.copy()
        sp[idx] += eps
        sm[idx] -= eps
        fd = (_loss(d.dY, d.X, phi0, sp, d.A, d.B, layer) - _loss(d.dY, d.X, phi0, sm, d.A, d.B, layer)) / (2 * eps)
        assert abs(fd - g["ds"][idx]) <= 1e-9 * max(1.0, abs(fd))


def test_adapter_gradients_equal_surrogate_autograd():
    """Where no element is clipped (M = 1), the STE gradients w.r.t. A and B are the
    exact gradients of the smooth surrogate s * (phi^{-1}(Phi0) + (alpha/r) A B)."""
    torch = pytest.importorskip("torch")
    layer = O.Layer(m=8, k=16, r=4, alpha=2.0, bits=4)
    spec = WL.LayerSpec("t", 8, 16, 4, 2.0, 4, 0, WL.PHI_QFIXED, a_std=0.1, b_std=0.1)
    d = WL.make_layer(spec, 5, seed=17)
    s0 = O.minmax_scale(d.W0, layer) * np.float32(1.5)       # wide range: nothing clips
    phi0 = O.downcast(d.W0, s0, layer)
    g = O.linear_bwd(d.dY, d.X, phi0, s0, d.A, d.B, layer)
    assert g["fq"]["M"].min() == 1.0
    P = torch.tensor(O.upcast(phi0, layer), dtype=torch.float64)
    A = torch.tensor(d.A, dtype=torch.float64, requires_grad=True)
    B = torch.tensor(d.B, dtype=torch.float64, requires_grad=True)
    s = torch.tensor(s0, dtype=torch.float64)[:, None]
    W = s * (P + (layer.alpha / layer.r) * (A @ B))
    loss = (torch.tensor(d.dY, dtype=torch.float64) * (torch.tensor(d.X, dtype=torch.float64) @ W.T)).sum()
    loss.backward()
    np.testing.assert_allclose(g["dA"], A.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(g["dB"], B.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_workload_generator_is_deterministic_and_bf16_exact():
    spec = WL.workload("tiny").layers[0]
    a = WL.make_layer(spec, 64, seed=0)
    b = WL.make_layer(spec, 64, seed=0)
    for name in ("W0", "A_bits", "B_bits", "X_bits", "dY_bits"):
        np.testing.assert_array_equal(getattr(a, name), getattr(b, name))
    # bf16 values widen exactly and re-round to the same bits
    np.testing.assert_array_equal(WL.bf16_bits(a.X), a.X_bits)
    assert WL.bf16_bits(np.array([1.0 + 2.0 ** -8], dtype=np.float32))[0] == 0x3F80   # tie -> even
    assert WL.bf16_bits(np.array([1.0 + 3 * 2.0 ** -8], dtype=np.float32))[0] == 0x3F82


# ---------------------------------------------------------------------------
# Asymmetric weights with a frozen zero offset (INT2 runs of Sec. 4; Eq. 1 with
# the offset outside the rounding, end of Sec. 3; reading R13)
# ---------------------------------------------------------------------------
def _asym_data(bits, phi, group=0, m=24, k=256, r=4, T=1, seed=7, std=0.01, zero_B=False):
    """A layer whose rows are shifted by different offsets, so that the zero
    offsets z0 of min-max range setting spread over the grid."""
    layer = O.Layer(m, k, r, float(r), bits, group, phi)
    spec = WL.LayerSpec("t", m, k, r, float(r), bits, group, phi, a_std=std, b_std=std)
    d = WL.make_layer(spec, T, seed=seed, zero_B=zero_B)
    rng = np.random.default_rng(seed + 100)
    shift = rng.uniform(-0.05, 0.05, size=(m, 1)).astype(np.float32)
    W0 = (d.W0 + shift).astype(np.float32)
    return layer, d, W0


@pytest.mark.parametrize("bits,phi,group", [(2, O.PHI_QFIXED, 0), (2, O.PHI_INT_PACKED, 128),
                                            (3, O.PHI_INT_PACKED, 0), (4, O.PHI_QFIXED, 128)])
def test_asym_minmax_range_covers_min_and_max(bits, phi, group):
    """s0 = (max - min) / (2^b - 1) and z0 = round(n - min / s0): the dequantized grid
    s0 (j - z0), j in [n, p], reaches min and max to within half a step."""
    layer, _, W0 = _asym_data(bits, phi, group)
    n, p = O.grid(bits)
    s0, z0 = O.minmax_range_asym(W0, layer)
    seg = W0.reshape(layer.m, -1, group if group else layer.k)
    lo, hi = seg.min(axis=2).reshape(s0.shape), seg.max(axis=2).reshape(s0.shape)
    np.testing.assert_array_equal(s0, np.float32(hi - lo) / np.float32(2 ** bits - 1))
    assert np.all(z0 == np.rint(z0)) and z0.min() >= n and z0.max() <= p
    assert len(np.unique(z0)) > 1                                  # the offsets really vary
    inner = (z0 > n) & (z0 < p)                                    # z0 not clipped
    step = s0.astype(np.float64)
    assert np.all(np.abs(step * (n - z0) - lo)[inner] <= 0.5 * step[inner] * (1 + 1e-6))
    assert np.all(np.abs(step * (p - z0) - hi)[inner] <= 0.5 * step[inner] * (1 + 1e-6))


@pytest.mark.parametrize("bits,group", [(2, 0), (2, 128), (3, 0), (4, 128)])
def test_asym_int_phi_with_zero_adapter_is_asymmetric_rtn(bits, group):
    """phi = INT-b and A B = 0: W_Z is Eq. 1's clip(round(W0 / s0) + z0, n, p), taken
    here in that order (round first, then add z0), and s0 (W_Z - z0) is Eq. 1's
    dequantized W0."""
    layer, d, W0 = _asym_data(bits, O.PHI_INT_PACKED, group, zero_B=True)
    n, p = O.grid(bits)
    s0, z0 = O.minmax_range_asym(W0, layer)
    x32 = np.divide(W0, O.expand_scale(s0, layer).astype(np.float32), dtype=np.float32)
    zf = O.expand_scale(z0, layer)
    expect = np.clip(_rtn_python(x32, -10 ** 6, 10 ** 6) + zf, n, p)
    phi0 = O.downcast(W0, s0, layer, z0)
    wz = O.merge(phi0, d.A, d.B, layer).astype(np.int64)
    np.testing.assert_array_equal(wz, expect)
    fq = O.fake_quant_weight(phi0, s0, d.A, d.B, layer, z0)
    np.testing.assert_array_equal(fq["W_hat"], O.expand_scale(s0, layer) * (expect - zf))


def test_asym_zero_offsets_of_zero_reduce_to_symmetric():
    """z = 0 everywhere gives exactly the symmetric path (Eq. 8)."""
    layer, d, W0 = _asym_data(4, O.PHI_QFIXED, 0, T=3, std=0.3)
    s0 = O.minmax_scale(W0, layer)
    z0 = np.zeros_like(s0)
    phi_s, phi_a = O.downcast(W0, s0, layer), O.downcast(W0, s0, layer, z0)
    np.testing.assert_array_equal(phi_s, phi_a)
    gs = O.linear_bwd(d.dY, d.X, phi_s, s0, d.A, d.B, layer)
    ga = O.linear_bwd(d.dY, d.X, phi_a, s0, d.A, d.B, layer, None, z0)
    for name in ("dX", "dA", "dB", "ds"):
        np.testing.assert_array_equal(gs[name], ga[name], err_msg=name)


ASYM_LOOP_CASES = [
    dict(bits=2, phi=O.PHI_QFIXED, group=0, std=0.5),
    dict(bits=2, phi=O.PHI_INT_PACKED, group=0, std=1.0),
    dict(bits=3, phi=O.PHI_QFIXED, group=128, std=1.0),
]


@pytest.mark.parametrize("case", ASYM_LOOP_CASES)
def test_asym_ste_gradients_match_scalar_loops_and_finite_differences(case):
    """With zero offsets: the matrix-form gradients equal the hand-expanded loops, and
    dX and ds equal central differences of <dY, Y> (Y is linear in X and in s; the
    codes do not depend on s), while s (W_Z - z) reproduces W_hat."""
    layer, d, W0 = _asym_data(case["bits"], case["phi"], case["group"], m=4, k=256, r=2, T=3,
                              std=case["std"])
    s0, z0 = O.minmax_range_asym(W0, layer)
    phi0 = O.downcast(W0, s0, layer, z0)
    s = s0 * np.float32(0.9)
    ref = O.linear_bwd_loops(d.dY, d.X, phi0, s, d.A, d.B, layer, None, z0)
    got = O.linear_bwd(d.dY, d.X, phi0, s, d.A, d.B, layer, None, z0)
    for name in ("dX", "dA", "dB", "ds"):
        np.testing.assert_allclose(got[name], ref[name], rtol=1e-12, atol=1e-12, err_msg=name)
    assert got["fq"]["M"].min() == 0.0                              # the clip mask is exercised
    wz = O.merge(phi0, d.A, d.B, layer).astype(np.float64)
    np.testing.assert_array_equal(O.expand_scale(s, layer) * (wz - O.expand_scale(z0, layer)),
                                  got["fq"]["W_hat"])

    def loss(X, s_):
        return float(np.sum(d.dY * O.linear_fwd(X, phi0, s_, d.A, d.B, layer, None, z0)))
    eps = 0.5
    X64 = d.X.astype(np.float64)
    for (t, j) in [(0, 0), (2, layer.k - 1)]:
        Xp, Xm = X64.copy(), X64.copy()
        Xp[t, j] += eps
        Xm[t, j] -= eps
        fd = (loss(Xp, s) - loss(Xm, s)) / (2 * eps)
        assert abs(fd - got["dX"][t, j]) <= 1e-9 * max(1.0, abs(fd))
    s64 = s.astype(np.float64)
    for idx in [(0,) if s.ndim == 1 else (0, 0), (layer.m - 1,) if s.ndim == 1 else (layer.m - 1, 1)]:
        sp, sm = s64.copy(), s64.copy()
        sp[idx] += eps
        sm[idx] -= eps
        fd = (loss(X64, sp) - loss(X64, sm)) / (2 * eps)
        assert abs(fd - got["ds"][idx]) <= 1e-9 * max(1.0, abs(fd))


# ---------------------------------------------------------------------------
# Per-token activations (default of the weight-activation runs, Sec. 4; reading R14)
# ---------------------------------------------------------------------------
def test_per_token_absmax_scale_and_error_bound():
    """Each token's largest |X| lands on code +-127, nothing clips, and the rounding
    error of every element is at most half of its token's step."""
    rng = np.random.default_rng(31)
    X = (rng.standard_normal((40, 96)) * rng.uniform(0.01, 10.0, size=(40, 1))).astype(np.float32)
    X[7] = 0.0                                                      # an all-zero token
    codes, Xh, mask, s_x = O.act_quant_per_token(X)
    assert s_x[7] == 1.0 and np.all(codes[7] == 0)
    live = np.arange(40) != 7
    assert np.all(np.abs(codes[live]).max(axis=1) == 127)
    assert mask.min() == 1.0
    err = np.abs(Xh - X.astype(np.float64))
    assert np.all(err <= 0.5 * s_x.astype(np.float64)[:, None] * (1 + 1e-6))


def test_per_token_equals_per_tensor_for_equal_token_ranges():
    """When every token has the same absmax, the per-token quantizer is the per-tensor
    one (Eq. 1, z = 0) with that scale."""
    rng = np.random.default_rng(32)
    X = rng.standard_normal((12, 64)).astype(np.float32)
    X /= np.abs(X).max(axis=1, keepdims=True)                       # every token's absmax is 1
    X = (X * np.float32(3.0)).astype(np.float32)
    c1, Xh1, m1, s_x = O.act_quant_per_token(X)
    assert np.all(s_x == s_x[0])
    c2, Xh2, m2 = O.act_quant(X, float(s_x[0]))
    np.testing.assert_array_equal(c1, c2)
    np.testing.assert_array_equal(Xh1, Xh2)


def test_per_token_ste_gradients_match_scalar_loops():
    layer = O.Layer(4, 6, 2, 2.0, 4, 0, O.PHI_QFIXED, 8, True)
    spec = WL.LayerSpec("t", 4, 6, 2, 2.0, 4, 0, WL.PHI_QFIXED, a_std=0.5, b_std=0.5)
    d = WL.make_layer(spec, 5, seed=19)
    s0 = O.minmax_scale(d.W0, layer)
    phi0 = O.downcast(d.W0, s0, layer)
    ref = O.linear_bwd_loops(d.dY, d.X, phi0, s0, d.A, d.B, layer)
    got = O.linear_bwd(d.dY, d.X, phi0, s0, d.A, d.B, layer)
    for name in ("dX", "dA", "dB", "ds"):
        np.testing.assert_allclose(got[name], ref[name], rtol=1e-12, atol=1e-12, err_msg=name)
    Xh = O.act_quant_per_token(d.X)[1]
    np.testing.assert_allclose(O.linear_fwd(d.X, phi0, s0, d.A, d.B, layer),
                               Xh @ O.fake_quant_weight(phi0, s0, d.A, d.B, layer)["W_hat"].T, rtol=0, atol=0)


# ---------------------------------------------------------------------------
# Optimizer step (App. B, Table B1; reading R17)
# ---------------------------------------------------------------------------
def test_adamw_first_step_closed_form():
    """Step 1 without decay: m_hat = g, v_hat = g^2, so p moves by -lr g / (|g| + eps)."""
    rng = np.random.default_rng(41)
    p0, g = rng.standard_normal(50), rng.standard_normal(50)
    p1, m, v = O.adamw_update(p0, g, np.zeros(50), np.zeros(50), 1, lr=1e-3)
    np.testing.assert_allclose(p1, p0 - 1e-3 * g / (np.abs(g) + 1e-8), rtol=1e-13, atol=1e-16)
    np.testing.assert_allclose(m, 0.1 * g, rtol=1e-14)
    np.testing.assert_allclose(v, 0.05 * g * g, rtol=1e-14)


def test_clip_coefficient_cases():
    g1, g2 = np.full(4, 0.25), np.full(12, 0.0)                    # norm 0.5 <= 1: untouched
    assert O.clip_coefficient([g1, g2], 1.0) == 1.0
    g3 = np.array([3.0, 4.0])                                      # norm 5: scaled to ~1
    c = O.clip_coefficient([g3], 1.0)
    assert abs(c * 5.0 - 1.0) < 1e-6


def test_adamw_with_clipping_matches_torch_optimizer():
    """Three clipped AdamW steps on A, B, s (two parameter groups with their own
    learning rates, as in Table B1) agree with torch.optim.AdamW and
    torch.nn.utils.clip_grad_norm_, an independent implementation."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(42)
    shapes = {"A": (6, 3), "B": (3, 8), "s": (6,)}
    lrs = {"A": 1e-3, "B": 1e-3, "s": 1e-4}
    params = {k: rng.standard_normal(sh) for k, sh in shapes.items()}
    tp = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in params.items()}
    opt = torch.optim.AdamW([{"params": [tp["A"], tp["B"]], "lr": lrs["A"]}, {"params": [tp["s"]], "lr": lrs["s"]}],
                            betas=(0.9, 0.95), eps=1e-8, weight_decay=0.0)
    state = {k: (np.zeros(sh), np.zeros(sh)) for k, sh in shapes.items()}
    for step in range(1, 4):
        grads = {k: rng.standard_normal(sh) * (3.0 if step == 2 else 0.1) for k, sh in shapes.items()}
        coef = O.clip_coefficient(list(grads.values()), 1.0)
        for k in shapes:
            params[k], m, v = O.adamw_update(params[k], coef * grads[k], *state[k], step, lrs[k])
            state[k] = (m, v)
        opt.zero_grad()
        for k in shapes:
            tp[k].grad = torch.tensor(grads[k], dtype=torch.float64)
        torch.nn.utils.clip_grad_norm_([tp[k] for k in shapes], 1.0)
        opt.step()
        for k in shapes:
            np.testing.assert_allclose(params[k], tp[k].detach().numpy(), rtol=1e-12, atol=1e-15, err_msg=f"{k} {step}")
    assert O.clip_coefficient([rng.standard_normal(10) * 3.0], 1.0) < 1.0    # clipping path was reachable


# ---------------------------------------------------------------------------
# L^p range setting (App. B; reading R18)
# ---------------------------------------------------------------------------
def test_lp_range_brute_force_and_properties():
    """On a tiny layer the chosen scale is the brute-force minimiser over the candidate
    grid (written independently, with Python's round), the last candidate is min-max
    itself, and a row with an outlier clips it under L2 (a scale below min-max)."""
    layer = O.Layer(4, 64, 2, 2.0, 3, 0, O.PHI_QFIXED)
    rng = np.random.default_rng(51)
    W0 = (rng.standard_normal((4, 64)) * 0.02).astype(np.float32)
    W0[1, 5] = 0.3                                                  # an outlier row
    s_mm = O.minmax_scale(W0, layer)
    cands = O.lp_candidates(s_mm, 100)
    assert np.all(cands[:, -1] == s_mm)
    s2, j2 = O.lp_range(W0, layer, 2.0)
    n, p = O.grid(3)
    for i in range(4):
        # brute force written independently: quantize-dequantize for every candidate
        best, best_j = None, None
        for j in range(100):
            s = float(cands[i, j])
            q = np.array([min(max(round(float(np.float32(w) / np.float32(s))), n), p) for w in W0[i]], dtype=np.float64)
            loss = float(np.sum((W0[i].astype(np.float64) - s * q) ** 2))
            if best is None or loss < best:
                best, best_j = loss, j
        assert j2[i] == best_j, (i, j2[i], best_j)
    assert s2[1] < s_mm[1]                                          # the outlier row clips its outlier under L2


def test_lp_range_groups_shape():
    layer = O.Layer(2, 256, 2, 2.0, 4, 128, O.PHI_QFIXED)
    W0 = (np.random.default_rng(52).standard_normal((2, 256)) * 0.02).astype(np.float32)
    s0, j = O.lp_range(W0, layer, 2.4, n_cand=40)
    assert s0.shape == (2, 2) and j.shape == (2, 2)
    assert np.all(s0 <= O.minmax_scale(W0, layer))


# ---------------------------------------------------------------------------
# Floating-point downcasting operators (Sec. 3; reading R19)
# ---------------------------------------------------------------------------
FP8_TORCH = [(O.PHI_FP8_E4M3, "float8_e4m3fn", 448.0), (O.PHI_FP8_E5M2, "float8_e5m2", 57344.0)]


@pytest.mark.parametrize("fmt,tname,vmax", FP8_TORCH)
def test_fp8_decode_exhaustive_against_torch(fmt, tname, vmax):
    """All 256 FP8 patterns decode (from the format definition) to torch's values; the
    non-finite patterns are exactly torch's; the largest finite value is the format's."""
    torch = pytest.importorskip("torch")
    td = getattr(torch, tname, None)
    if td is None:
        pytest.skip(f"torch has no {tname}")
    codes = np.arange(256, dtype=np.uint8)
    ours = O.fp8_decode(codes, fmt)
    ref = torch.from_numpy(codes).view(td).to(torch.float64).numpy()
    fin = np.isfinite(ref)
    np.testing.assert_array_equal(ours[fin], ref[fin])
    assert np.all(np.isnan(ours[~fin]))
    assert np.nanmax(ours) == vmax and np.nanmin(ours) == -vmax


@pytest.mark.parametrize("fmt,tname,vmax", FP8_TORCH)
def test_fp8_encode_against_torch_midpoints_and_saturation(fmt, tname, vmax):
    """In range the cast equals torch's round-to-nearest-even cast bit for bit (signed
    zeros included); every finite pattern round-trips; an exact midpoint between two
    neighbours takes the even pattern; beyond the largest finite value it saturates."""
    torch = pytest.importorskip("torch")
    td = getattr(torch, tname, None)
    if td is None:
        pytest.skip(f"torch has no {tname}")
    rng = np.random.default_rng(61)
    x = (rng.standard_normal(200000) * 10.0 ** rng.uniform(-4, np.log10(vmax) - 0.5, 200000)).astype(np.float32)
    x = np.concatenate([x[np.abs(x) <= vmax], np.float32([0.0, -0.0, 1e-30, -1e-30])])   # torch does not saturate
    ref = torch.from_numpy(x).to(td).view(torch.uint8).numpy()
    np.testing.assert_array_equal(O.fp8_encode(x, fmt), ref)
    vals = O.fp8_decode(np.arange(256, dtype=np.uint8), fmt)
    finite = np.nonzero(np.isfinite(vals))[0].astype(np.uint8)
    np.testing.assert_array_equal(O.fp8_encode(vals[finite].astype(np.float32), fmt), finite)
    pos = np.nonzero(np.isfinite(vals[:128]))[0]
    mids = ((vals[pos[:-1]] + vals[pos[1:]]) / 2).astype(np.float32)     # exact in fp32
    got = O.fp8_encode(mids, fmt)
    assert np.all(got % 2 == 0)
    assert np.all((got == pos[:-1]) | (got == pos[1:]))
    big = np.float32([vmax * 1.01, 1e30, -1e30])
    np.testing.assert_array_equal(O.fp8_decode(O.fp8_encode(big, fmt), fmt), [vmax, vmax, -vmax])


def test_bf16_and_fp16_casts_against_torch():
    """bf16 (written from the bit pattern) and fp16 casts equal torch's casts, including
    constructed exact midpoints, which go to the even neighbour; bf16_round of an fp32
    value is the same rounding."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(62)
    x = (rng.standard_normal(100000) * 10.0 ** rng.uniform(-6, 3, 100000)).astype(np.float32)
    mid = ((rng.integers(0, 1 << 15, 1000, dtype=np.uint32) << 16) | 0x8000).astype(np.uint32).view(np.float32)
    mid = mid[np.isfinite(mid) & (np.abs(mid) < 1e30) & (np.abs(mid) > 1e-37)]   # bf16's normal range
    for v in (x, mid):
        np.testing.assert_array_equal(O.float_cast(v, O.PHI_BF16),
                                      torch.from_numpy(v).bfloat16().view(torch.int16).numpy().view(np.uint16))
        np.testing.assert_array_equal(O.bf16_round(v.astype(np.float64)), O.bf16_decode(O.bf16_encode(v)))
    np.testing.assert_array_equal(O.bf16_encode(mid) & 1, 0)
    x16 = x[np.abs(x) <= 65504.0]
    np.testing.assert_array_equal(O.float_cast(x16, O.PHI_FP16),
                                  torch.from_numpy(x16).half().view(torch.int16).numpy().view(np.uint16))
    sat = O.float_value(O.float_cast(np.float32([7e4, -1e30]), O.PHI_FP16), O.PHI_FP16)
    np.testing.assert_array_equal(sat, [65504.0, -65504.0])


# format, bound on the relative cast error: half a unit in the last place, 2^-s for
# s significant bits (bf16 8, fp16 11, E4M3 4, E5M2 3)
FLOAT_PHI_ERR = [(O.PHI_BF16, 2.0 ** -8), (O.PHI_FP16, 2.0 ** -11), (O.PHI_FP8_E4M3, 2.0 ** -4),
                 (O.PHI_FP8_E5M2, 2.0 ** -3)]


@pytest.mark.parametrize("fmt,rel", FLOAT_PHI_ERR)
def test_float_phi_with_zero_adapter_is_rtn_near_ties_aside(fmt, rel):
    """phi = a floating-point cast and B = 0: W_Z equals round-to-nearest quantization
    of W0 (Python's round) except on elements within the cast's half-ulp of a
    half-integer, where the cast may move x across or onto it; the stored value is
    within that bound of x and never clipped inside phi."""
    bits = 4
    layer = O.Layer(m=64, k=128, r=4, alpha=4.0, bits=bits, phi_format=fmt)
    spec = WL.LayerSpec("t", 64, 128, 4, 4.0, bits, 0, fmt, outlier_frac=0.01)
    d = WL.make_layer(spec, 1, seed=63, zero_B=True, with_activations=False)
    s0 = O.minmax_scale(d.W0, layer) * np.float32(0.5)       # half range: phi must keep |x| > p
    x32 = np.divide(d.W0, s0[:, None].astype(np.float32), dtype=np.float32)
    phi0 = O.downcast(d.W0, s0, layer)
    stored = O.upcast(phi0, layer)
    x = x32.astype(np.float64)
    sub = 2.0 ** -10 if fmt in (O.PHI_FP8_E4M3, O.PHI_FP8_E5M2) else 0.0    # half the E4M3 subnormal step
    assert np.all(np.abs(stored - x) <= rel * np.abs(x) + sub)
    n, p = O.grid(bits)
    assert np.abs(stored).max() > p                            # no clip inside phi
    wz = O.merge(phi0, d.A, d.B, layer).astype(np.int64)
    rtn = _rtn_python(x32, n, p)
    near = np.abs(x - (np.floor(x) + 0.5)) <= rel * np.abs(x) + sub
    assert np.all((wz == rtn) | near)


def test_float_phi_rejects_zero_offsets():
    layer = O.Layer(m=2, k=4, r=1, alpha=1.0, bits=2, phi_format=O.PHI_BF16)
    with pytest.raises(ValueError):
        O.downcast(np.ones((2, 4), np.float32), np.ones(2, np.float32), layer, np.zeros(2, np.float32))


# ---------------------------------------------------------------------------
# bf16 pre-round value (reading R20): what the R2 choice changes
# ---------------------------------------------------------------------------
def test_bf16_u_matches_exact_u_where_nothing_rounds():
    """With B = 0 and a base that bf16 holds exactly (Q4.4: at most 8 significant bits;
    phi = BF16), every bf16 rounding of R20 is exact: the codes equal R2's."""
    for fmt in (O.PHI_QFIXED, O.PHI_BF16):
        layer = O.Layer(m=32, k=64, r=4, alpha=4.0, bits=4, phi_format=fmt)
        spec = WL.LayerSpec("t", 32, 64, 4, 4.0, 4, 0, fmt, outlier_frac=0.01)
        d = WL.make_layer(spec, 1, seed=64, zero_B=True, with_activations=False)
        s0 = O.minmax_scale(d.W0, layer)
        phi0 = O.downcast(d.W0, s0, layer)
        lay16 = O.Layer(32, 64, 4, 4.0, 4, 0, fmt, u_bf16=True)
        np.testing.assert_array_equal(O.merge(phi0, d.A, d.B, lay16), O.merge(phi0, d.A, d.B, layer))


def test_bf16_u_swallows_small_adapter_updates():
    """A bf16 u cannot move a base value in [2, 4) by less than half its ulp (2^-7):
    there the R20 code is round(phi^{-1}(Phi0)) whatever A B adds, while the exact u of
    R2 lets the same update flip codes that sit on a half-integer (Q4.4 stores 2.5)."""
    layer = O.Layer(m=1, k=8, r=1, alpha=1.0, bits=4)
    lay16 = O.Layer(1, 8, 1, 1.0, 4, u_bf16=True)
    P = np.array([[2.5, -2.5, 3.5, -3.5, 2.0625, 3.9375, -2.4375, 2.5]])
    phi0 = (P * 16).astype(np.int8)
    A = np.ones((1, 1))
    B = np.array([[2.0 ** -8, 2.0 ** -8, -2.0 ** -8, 2.0 ** -8, 2.0 ** -9, -2.0 ** -9, 2.0 ** -8, -2.0 ** -8]])
    np.testing.assert_array_equal(O.merge(phi0, A, B, lay16)[0], np.clip(np.rint(P[0]), -8, 7))
    exact = O.merge(phi0, A, B, layer)[0]
    np.testing.assert_array_equal(exact, [3, -2, 3, -3, 2, 4, -2, 2])


# ---------------------------------------------------------------------------
# Reading R8: the downcast divides in fp32; which codes a float64 division would move
# ---------------------------------------------------------------------------
def _fl32_exact(q):
    """The fp32 value nearest to the rational q, ties to even (checked against both
    neighbours of a first guess in exact arithmetic)."""
    from fractions import Fraction
    c = np.float32(float(q))
    cands = [np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))]
    best = min(cands, key=lambda v: (abs(Fraction(float(v)) - q), int(np.float32(v).view(np.uint32)) & 1))
    return Fraction(float(best))


def test_fp64_division_changes_match_exact_arithmetic():
    """Weights built to put W0 / s0 next to rounding boundaries of Q4.4 (x = (j + 1/2)/16)
    and of INT-4 (x = j + 1/2), with their fp32 neighbours: the oracle's mask of elements whose base changes under a
    float64 division equals the one found with exact rationals (the fp32 quotient as the
    correctly rounded fp32 of W0 / s0, the float64 one as Python's correctly rounded float),
    and it is not empty."""
    from fractions import Fraction
    s0 = np.float32(0.3)
    for fmt, step in ((O.PHI_QFIXED, 16), (O.PHI_INT_PACKED, 1)):
        js = np.arange(-120, 112) if step == 16 else np.arange(-8, 7)
        mid = np.array([np.float32(float(s0) * (j + 0.5) / step) for j in js], dtype=np.float32)
        vals = np.concatenate([mid, np.nextafter(mid, np.float32(np.inf)), np.nextafter(mid, np.float32(-np.inf))])
        k = len(vals) + (-len(vals)) % 16
        W0 = np.zeros((1, k), dtype=np.float32)
        W0[0, :len(vals)] = vals
        layer = O.Layer(1, k, 1, 1.0, 4, 0, fmt)
        got = O.downcast_fp64_changes(W0, np.array([s0]), layer)[0]
        n, p = O.grid(4)
        want = np.zeros(k, dtype=bool)
        for i, w in enumerate(W0[0]):
            q = Fraction(float(w)) / Fraction(float(s0))
            codes = []
            for x in (_fl32_exact(q), Fraction(float(q))):
                x = min(max(x, n), p)
                y = x * step
                r = round(y)                       # Python's round: half to even, exact on Fractions
                codes.append(r)
            want[i] = codes[0] != codes[1]
        np.testing.assert_array_equal(got, want)
        assert want.sum() > 0
