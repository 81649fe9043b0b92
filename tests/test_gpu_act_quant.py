"""GPU parity of the activation quantizer (the int8 fake quantizer of the
weight-activation runs, Eq. 1 with z = 0, b = 8) on its own, bit for bit against
the oracle: per tensor the codes and the clip-mask bits, per token X_hat = bf16(s_x[t]
X_Z).  Token counts leave ragged 32-token mask words; scales small enough to clip."""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import bits_to_f32, to_dev, torch

pytestmark = pytest.mark.gpu


def _layer(k, per_token):
    spec = WL.LayerSpec("aq", 128, k, 4, 4.0, 4, 0, WL.PHI_QFIXED, 8, act_per_token=per_token)
    return LQ.Layer.from_spec(spec)


def _x(T, k, seed):
    rng = np.random.default_rng(seed)
    X = (rng.standard_normal((T, k)) * 10.0 ** rng.uniform(-1, 1, (T, 1))).astype(np.float32)
    X[rng.random((T, k)) < 1e-3] *= 20.0      # outliers
    bits = WL.bf16_bits(X)
    return bits, WL.bf16_to_f32(bits)


@pytest.mark.parametrize("T,k,sx_factor", [(1, 128, 1.0), (31, 384, 0.3), (33, 128, 1.0), (1000, 512, 0.05),
                                           (257, 4096, 0.5)])
def test_per_tensor_codes_and_mask_bit_exact(T, k, sx_factor):
    t = torch()
    bits, X = _x(T, k, seed=T + k)
    s_x_host = np.float32(np.float32(np.abs(X).max()) / np.float32(127.0) * np.float32(sx_factor))
    s_x = t.tensor([s_x_host], dtype=t.float32, device="cuda")
    out = t.empty((T, k), dtype=t.int16, device="cuda")
    words = (T + 31) // 32
    mask = t.full((k, words), -1, dtype=t.int32, device="cuda")
    LQ.act_quant(_layer(k, False), T, to_dev(bits), s_x, out, mask)
    LQ.get_device_status()
    codes, _, M = O.act_quant(X, s_x_host)
    np.testing.assert_array_equal(bits_to_f32(out), codes)
    got = mask.cpu().numpy().view(np.uint32)
    ref = np.zeros((k, words), dtype=np.uint32)
    for tt in range(T):
        ref[:, tt // 32] |= (M[tt].astype(np.uint32) << np.uint32(tt % 32))
    np.testing.assert_array_equal(got, ref)
    if sx_factor < 1.0:
        assert M.min() == 0.0                 # some values clip


@pytest.mark.parametrize("T,k", [(1, 128), (5, 384), (300, 4096), (7, 16384), (3, 16512)])
def test_per_token_x_hat(T, k):
    """X_hat = bf16(s_x[t] X_Z): the codes equal the oracle's exactly; the bf16 value is the
    nearest to the exact product except where the fp32 product sits on a bf16 midpoint
    (one rounding in the oracle's reading, fp32 then bf16 on the device); a zero token
    gets the unit scale and zero codes.  k = 16512 takes the rereading kernel."""
    t = torch()
    bits, X = _x(T, k, seed=3 * T + k)
    if T > 2:
        bits[2, :] = 0
        X[2, :] = 0.0
    out = t.empty((T, k), dtype=t.int16, device="cuda")
    LQ.act_quant(_layer(k, True), T, to_dev(bits), None, out)
    LQ.get_device_status()
    codes, _, _, s_x = O.act_quant_per_token(X)
    exact = s_x.astype(np.float64)[:, None] * codes
    got = bits_to_f32(out).astype(np.float64)
    ref = O.bf16_round(np.where(exact == 0, 1.0, exact)) * (exact != 0)
    prod32 = (s_x[:, None] * codes.astype(np.float32)).astype(np.float32).astype(np.float64)
    on_mid = O.bf16_round(prod32 * (1 + 2.0 ** -30)) != O.bf16_round(prod32 * (1 - 2.0 ** -30))
    assert ((got != ref) & ~on_mid).sum() == 0
    assert np.all(np.abs(got - exact) <= np.abs(exact) * 2.0 ** -8 + 1e-30)
    if T > 2:
        assert np.all(got[2] == 0)
