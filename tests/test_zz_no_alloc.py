"""The allocation-free forward, lrqat_linear_fwd_noalloc, called through the C ABI.

Some callers cannot allocate device memory (runtimes that own all device memory
and give an operator only its inputs and outputs, or that forbid allocation after
start-up because cudaMalloc can synchronize the device); this entry point serves
them from a fixed scratch array inside the library.  The cases below make the
forward use that array: a rank that is not a multiple of 8 (the adapters are
copied into padded layouts there), per-tensor int8 activations (their codes
live there) and a group-wise layer on CTA pairs (its scales go there as bf16
rows).  Each output must equal the workspace-based lrqat_linear_fwd's bit for
bit (the same kernels read the same operands) and the oracle's within the
forward tolerance, on calls in a row with different layers (each call reuses the
scratch the previous one left behind), and layers whose scratch does not fit must
be rejected cleanly.

This file is collected last on purpose, so that a run which stops at the first
failure has already run every other test.
"""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL
from paper_2406_06385_gb300.build import build

from gpu_util import DeviceLayer, bits_to_f32, oracle_layer, to_dev, torch

pytestmark = pytest.mark.gpu

TOL_Y = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _library():
    build()
    LQ.lib()


def _spec(name, m, k, r, bits=4, phi=WL.PHI_QFIXED, group=0, act=0):
    return WL.LayerSpec(name, m, k, r, float(r), bits, group, phi, act, outlier_frac=1e-3, a_std=0.2, b_std=0.2)


def _forward_both(spec, T, seed):
    """(no-alloc output, workspace output, oracle output) of one layer as fp32 arrays."""
    t = torch()
    data = WL.make_layer(spec, T, seed=seed)
    dl = DeviceLayer(data)
    X = to_dev(data.X_bits)
    L = dl.layer
    s_x, s_x_host = None, None
    if spec.act_bits == 8:
        s_x_host = float(np.float32(np.abs(data.X).max()) / np.float32(127.0) * np.float32(0.7))   # some codes clip
        s_x = t.tensor([s_x_host], dtype=t.float32, device="cuda")
    assert LQ.fwd_workspace_bytes(L, T) <= (4 << 20)
    y_ref = t.empty((T, spec.m), dtype=t.int16, device="cuda")
    ws = t.empty(LQ.fwd_workspace_bytes(L, T), dtype=t.uint8, device="cuda")
    LQ.linear_fwd(L, T, X, dl.phi0, dl.s, dl.A, dl.B, s_x, y_ref, ws)
    y_na = t.full((T, spec.m), 0x7FC0, dtype=t.int16, device="cuda")   # bf16 NaN everywhere beforehand
    LQ.linear_fwd_noalloc(L, T, X, dl.phi0, dl.s, dl.A, dl.B, s_x, y_na)
    LQ.get_device_status()
    OL = oracle_layer(spec)
    s0 = O.minmax_scale(data.W0, OL)
    y_or = O.linear_fwd(data.X, O.downcast(data.W0, s0, OL), s0, data.A, data.B, OL, s_x_host)
    return bits_to_f32(y_na), bits_to_f32(y_ref), y_or


def test_noalloc_forward_matches_workspace_forward_on_calls_in_a_row(lowrank_path):
    # the allocation-free forward computes the low-rank tile inside the GEMM; the workspace
    # forward is held to the same path, so the two are bit-identical
    lowrank_path("tile")
    cases = [
        (_spec("na_r20", 256, 512, 20), 1000, 31),                                   # padded adapters in the scratch
        (_spec("na_a8", 384, 512, 32, act=8), 1500, 32),                             # int8 codes in the scratch
        (_spec("na_r12_int3", 256, 768, 12, bits=3, phi=WL.PHI_INT_PACKED), 513, 33),
        (_spec("na_g128", 256, 512, 32, group=128), 700, 34),                        # scale rows in the scratch
        (_spec("na_r20", 256, 512, 20), 1000, 31),                                   # the first call again
    ]
    for spec, T, seed in cases:
        got, ref, orc = _forward_both(spec, T, seed)
        assert np.isfinite(got).all(), spec.name
        np.testing.assert_array_equal(got, ref, err_msg=spec.name)
        err = O.rel_fro(got, orc)
        assert err <= TOL_Y, (spec.name, err)


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
