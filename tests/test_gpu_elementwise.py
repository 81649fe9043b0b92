"""GPU parity of the memory-bound entry points: range setting, downcast and
merge, bit-exact against the oracle (merge: except near-tie elements)."""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import DeviceLayer, oracle_layer, phi_buffer, phi_host, to_dev, torch

pytestmark = pytest.mark.gpu

CASES = [
    # name, m, k, r, bits, group, phi, a_std, b_std
    ("q44_pc", 384, 512, 4, 4, 0, WL.PHI_QFIXED, 0.05, 0.05),
    ("q35_pc_rank32", 256, 384, 32, 3, 0, WL.PHI_QFIXED, 1 / 64, 1e-3),
    ("q44_g128", 256, 640, 16, 4, 128, WL.PHI_QFIXED, 0.05, 0.05),
    ("int3_packed", 384, 256, 32, 3, 0, WL.PHI_INT_PACKED, 0.1, 0.1),
    ("int4_packed_g256", 128, 512, 8, 4, 256, WL.PHI_INT_PACKED, 0.1, 0.1),
    ("q26_clip_heavy", 128, 256, 64, 2, 0, WL.PHI_QFIXED, 1.0, 1.0),
    ("q71", 128, 128, 1, 7, 0, WL.PHI_QFIXED, 0.05, 0.05),
    ("bf16_pc", 256, 512, 8, 4, 0, WL.PHI_BF16, 0.05, 0.05),
    ("fp16_g128_w3", 128, 640, 16, 3, 128, WL.PHI_FP16, 0.1, 0.1),
    ("fp8_e4m3_pc", 384, 256, 32, 4, 0, WL.PHI_FP8_E4M3, 0.1, 0.1),
    ("fp8_e5m2_g128_w2", 128, 512, 8, 2, 128, WL.PHI_FP8_E5M2, 0.3, 0.3),
    ("bf16_w8", 128, 256, 4, 8, 0, WL.PHI_BF16, 0.05, 0.05),
]


def _spec(c):
    name, m, k, r, bits, g, phi, a_std, b_std = c
    return WL.LayerSpec(name, m, k, r, float(r), bits, g, phi, outlier_frac=1e-3, a_std=a_std, b_std=b_std)


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_range_and_downcast_bit_exact(case):
    spec = _spec(case)
    data = WL.make_layer(spec, 1, seed=21, with_activations=False)
    dl = DeviceLayer(data)
    torch().cuda.synchronize()
    L = oracle_layer(spec)
    s0_ref = O.minmax_scale(data.W0, L)
    np.testing.assert_array_equal(dl.s0.cpu().numpy().reshape(s0_ref.shape), s0_ref)
    phi_ref = O.downcast(data.W0, s0_ref, L)
    got = dl.phi0.cpu().numpy()
    np.testing.assert_array_equal(got.view(phi_ref.dtype), phi_ref)


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_merge_matches_oracle_codes(case):
    spec = _spec(case)
    data = WL.make_layer(spec, 1, seed=22, with_activations=False)
    dl = DeviceLayer(data)
    wz = torch().empty((spec.m, spec.k), dtype=torch().int8, device="cuda")
    LQ.merge(dl.layer, dl.phi0, dl.A, dl.B, wz)
    LQ.get_device_status()
    L = oracle_layer(spec)
    phi_ref = phi_host(dl.phi0, spec)
    ones = np.ones((spec.m, spec.k // spec.group_size) if spec.group_size else (spec.m,))
    fq = O.fake_quant_weight(phi_ref, ones, data.A, data.B, L)
    ref = fq["c"].astype(np.int8)
    got = wz.cpu().numpy()
    n, p = O.grid(spec.bits)
    assert got.min() >= n and got.max() <= p
    exempt = O.near_tie(fq["u"])
    bad = (got != ref) & ~exempt
    assert bad.sum() == 0, f"{bad.sum()} code mismatches outside near-ties (near-ties: {exempt.sum()})"


def test_zero_row_gets_unit_scale_and_zero_codes():
    spec = WL.LayerSpec("z", 128, 256, 4, 4.0, 4, 0, WL.PHI_QFIXED)
    data = WL.make_layer(spec, 1, seed=3, with_activations=False)
    data.W0[5, :] = 0.0
    dl = DeviceLayer(data)
    s0 = dl.s0.cpu().numpy()
    assert s0[5] == 1.0
    assert np.all(dl.phi0.cpu().numpy()[5] == 0)


ASYM_CASES = [
    # id, m, k, bits, group, phi
    ("int2_q26_pc", 128, 256, 2, 0, WL.PHI_QFIXED),
    ("int2_packed_g128", 256, 512, 2, 128, WL.PHI_INT_PACKED),
    ("int3_packed_pc", 128, 384, 3, 0, WL.PHI_INT_PACKED),
    ("q44_g256", 128, 512, 4, 256, WL.PHI_QFIXED),
]


@pytest.mark.parametrize("case", ASYM_CASES, ids=[c[0] for c in ASYM_CASES])
def test_asym_range_and_downcast_bit_exact(case):
    """Asymmetric min-max range setting (s0 and zero offsets z0) and the downcast
    phi(W0 / s0 + z0) match the oracle exactly; the offsets really vary."""
    name, m, k, bits, g, phi = case
    spec = WL.LayerSpec(name, m, k, 4, 4.0, bits, g, phi, outlier_frac=1e-3, asym=True, w_row_shift=0.03)
    data = WL.make_layer(spec, 1, seed=23, with_activations=False)
    dl = DeviceLayer(data)
    torch().cuda.synchronize()
    L = oracle_layer(spec)
    s0_ref, z0_ref = O.minmax_range_asym(data.W0, L)
    np.testing.assert_array_equal(dl.s0.cpu().numpy().reshape(s0_ref.shape), s0_ref)
    np.testing.assert_array_equal(dl.z.cpu().numpy().reshape(z0_ref.shape), z0_ref)
    assert len(np.unique(z0_ref)) > 1
    phi_ref = O.downcast(data.W0, s0_ref, L, z0_ref)
    np.testing.assert_array_equal(dl.phi0.cpu().numpy().view(phi_ref.dtype), phi_ref)


LP_CASES = [
    # id, m, k, bits, group, p_norm, n_candidates
    ("q4_pc_p2.4", 128, 512, 4, 0, 2.4, 100),
    ("q3_g128_p3", 128, 640, 3, 128, 3.0, 100),
    ("q2_pc_p4", 128, 256, 2, 0, 4.0, 64),
    ("q4_g256_p2_n256", 128, 512, 4, 256, 2.0, 256),
    ("q4_long_row_p5", 128, 16384, 4, 0, 5.0, 100),    # 64 KB segment: opt-in shared memory
    ("q3_pc_p3.5_n1", 128, 256, 3, 0, 3.5, 1),
]


@pytest.mark.parametrize("case", LP_CASES, ids=[c[0] for c in LP_CASES])
def test_lp_range_matches_oracle(case):
    """L^p range setting: each scale is exactly one of the candidates fl32(s_max j / N);
    it is the oracle's choice, or (fp32 against fp64 losses) a candidate whose exact
    loss is within 1e-4 of the oracle's minimum; a zero row gets the first candidate
    of the unit scale, like min-max."""
    name, m, k, bits, g, p_norm, n_cand = case
    spec = WL.LayerSpec(name, m, k, 4, 4.0, bits, g, WL.PHI_QFIXED, outlier_frac=1e-3)
    data = WL.make_layer(spec, 1, seed=24, with_activations=False)
    data.W0[1, :] = 0.0
    dl = DeviceLayer(data)
    s0 = torch().empty_like(dl.s0)
    LQ.range_lp(dl.layer, dl.W0, s0, p_norm, n_cand)
    LQ.get_device_status()
    got = s0.cpu().numpy().reshape(m, -1)
    L = oracle_layer(spec)
    s0_ref, best_ref = O.lp_range(data.W0, L, p_norm, n_cand)
    s0_ref, best_ref = s0_ref.reshape(m, -1), best_ref.reshape(m, -1)
    cands = O.lp_candidates(O.minmax_scale(data.W0, L).reshape(m, -1), n_cand)
    segs = data.W0.reshape(m, got.shape[1], -1)
    n_diff = 0
    for i in range(m):
        for j in range(got.shape[1]):
            hit = np.nonzero(cands[i, j] == got[i, j])[0]
            assert hit.size >= 1, (i, j, got[i, j])
            if got[i, j] == s0_ref[i, j]:
                continue
            n_diff += 1
            ref_loss = O.lp_loss(segs[i, j], s0_ref[i, j], bits, p_norm)
            got_loss = O.lp_loss(segs[i, j], got[i, j], bits, p_norm)
            assert got_loss <= ref_loss * (1 + 1e-4), (i, j, got_loss, ref_loss)
    assert n_diff <= max(1, got.size // 20), n_diff
    assert np.all(got[1] == cands[1, :, 0]) and np.all(cands[1, :, 0] == np.float32(1.0 / n_cand))
    if n_cand > 1:
        assert len(np.unique(best_ref[2:])) > 1    # the search is not stuck at one end


@pytest.mark.parametrize("phi", [WL.PHI_FP8_E4M3, WL.PHI_FP8_E5M2, WL.PHI_BF16, WL.PHI_FP16])
def test_float_downcast_saturates_and_keeps_signed_zeros(phi):
    """Scales far below min-max push W0 / s0 beyond the FP8 and FP16 ranges: those casts
    saturate at the largest finite value; huge scales round small values to signed zeros
    (bf16 keeps them).  Bit for bit against the oracle."""
    t = torch()
    spec = WL.LayerSpec("sat", 128, 256, 4, 4.0, 4, 0, phi, outlier_frac=1e-3)
    data = WL.make_layer(spec, 1, seed=25, with_activations=False)
    L = oracle_layer(spec)
    lay = LQ.Layer.from_spec(spec)
    W0 = to_dev(data.W0)
    s_host = O.minmax_scale(data.W0, L).copy()
    s_host[: 64] *= np.float32(1e-4)       # |W0 / s| up to ~7e4: beyond E4M3 and E5M2
    s_host[64:] *= np.float32(1e12)        # |W0 / s| below every subnormal: signed zeros
    s_dev = t.from_numpy(s_host).cuda()
    phi0 = phi_buffer(spec)
    LQ.downcast(lay, W0, s_dev, phi0)
    LQ.get_device_status()
    ref = O.downcast(data.W0, s_host, L)
    np.testing.assert_array_equal(phi_host(phi0, spec), ref)
    if phi in (WL.PHI_FP8_E4M3, WL.PHI_FP8_E5M2):
        vmax = 448.0 if phi == WL.PHI_FP8_E4M3 else 57344.0
        assert np.abs(O.upcast(ref, L)[:64]).max() == vmax
    if phi != WL.PHI_BF16:
        small = O.upcast(ref, L)[64:]
        assert np.any((small == 0) & np.signbit(small)) and np.any((small == 0) & ~np.signbit(small))
