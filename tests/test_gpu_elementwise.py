"""GPU parity of the memory-bound entry points: range setting, downcast and
merge, bit-exact against the oracle (merge: except near-tie elements)."""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import DeviceLayer, oracle_layer, to_dev, torch

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
    phi_ref = dl.phi0.cpu().numpy().view(np.int8 if spec.phi_format == WL.PHI_QFIXED else np.uint8)
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
