"""The allocation-free forward, lrqat_linear_fwd_noalloc, called through the C ABI.

Some callers cannot allocate device memory (runtimes that own all device memory
and give an operator only its inputs and outputs, or that forbid allocation after
start-up because cudaMalloc can synchronize the device); this entry point serves
them from a fixed scratch array inside the library.  Its output must match the
workspace-based lrqat_linear_fwd within the forward tolerance, on two calls in a
row with different layers (the second call reuses the scratch the first one left
behind), and layers whose scratch does not fit must be rejected cleanly.

This file is collected last on purpose, so that a run which stops at the first
failure has already run every other test.
"""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL
from paper_2406_06385_gb300.build import build

from gpu_util import DeviceLayer, bits_to_f32, to_dev, torch

pytestmark = pytest.mark.gpu

TOL_Y = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _library():
    build()
    LQ.lib()


def _spec(name, m, k, r, bits=4, phi=WL.PHI_QFIXED, group=0, act=0):
    return WL.LayerSpec(name, m, k, r, float(r), bits, group, phi, act, outlier_frac=1e-3, a_std=0.2, b_std=0.2)


def _forward_both(spec, T, seed):
    t = torch()
    data = WL.make_layer(spec, T, seed=seed)
    dl = DeviceLayer(data)
    X = to_dev(data.X_bits)
    L = dl.layer
    y_ref = t.empty((T, spec.m), dtype=t.int16, device="cuda")
    ws = t.empty(LQ.fwd_workspace_bytes(L, T), dtype=t.uint8, device="cuda")
    LQ.linear_fwd(L, T, X, dl.phi0, dl.s, dl.A, dl.B, None, y_ref, ws)
    y_na = t.full((T, spec.m), 0x7FC0, dtype=t.int16, device="cuda")   # bf16 NaN everywhere beforehand
    LQ.linear_fwd_noalloc(L, T, X, dl.phi0, dl.s, dl.A, dl.B, None, y_na)
    LQ.get_device_status()
    return bits_to_f32(y_na), bits_to_f32(y_ref)


def test_noalloc_forward_matches_workspace_forward_on_two_calls_in_a_row():
    first = _forward_both(_spec("na1", 384, 512, 32), 1000, seed=31)
    second = _forward_both(_spec("na2", 256, 512, 16, bits=3, phi=WL.PHI_INT_PACKED), 513, seed=32)
    for got, ref in (first, second):
        assert np.isfinite(got).all()
        err = O.rel_fro(got, ref)
        assert err <= TOL_Y, err


def test_noalloc_forward_rejects_scratch_beyond_its_limit():
    t = torch()
    spec = _spec("big", 128, 4096, 8, act=8)
    L = LQ.Layer.from_spec(spec)
    T = 4096                                  # int8 activation codes alone need T * k * 2 = 32 MiB
    assert LQ.fwd_workspace_bytes(L, T) > (4 << 20)
    dummy = t.zeros(16, dtype=t.int16, device="cuda")
    s_x = t.ones(1, dtype=t.float32, device="cuda")
    with pytest.raises(LQ.LrqatError) as e:
        LQ.linear_fwd_noalloc(L, T, dummy, dummy, s_x, dummy, dummy, s_x, dummy)
    assert e.value.status == -4 and "fixed scratch" in str(e.value)
