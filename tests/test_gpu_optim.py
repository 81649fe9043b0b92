"""GPU parity of the optimizer step on A, B, s (App. B, Table B1): the global
gradient norm accumulated over layers and three clipped AdamW steps, against the
oracle (fp32 on the device, fp64 in the oracle)."""
import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import torch

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("group", [0, 128])
def test_clipped_adamw_matches_oracle(group):
    t = torch()
    rng = np.random.default_rng(7 + group)
    m, k, r = 256, 384, 8
    spec = WL.LayerSpec("opt", m, k, r, float(r), 4, group, WL.PHI_QFIXED)
    L = LQ.Layer.from_spec(spec)
    L_other = LQ.Layer.from_spec(WL.LayerSpec("other", 128, 128, 8, 8.0, 4, 0, WL.PHI_QFIXED))
    s_shape = (m, k // group) if group else (m,)
    A0 = WL.bf16_to_f32(WL.bf16_bits(rng.standard_normal((m, r)).astype(np.float32) * np.float32(0.02)))
    B0 = WL.bf16_to_f32(WL.bf16_bits(rng.standard_normal((r, k)).astype(np.float32) * np.float32(0.02)))
    s0 = rng.uniform(0.01, 0.02, size=s_shape).astype(np.float32)
    dev = lambda a: t.tensor(np.ascontiguousarray(a), device="cuda")
    A = dev(WL.bf16_bits(A0).view(np.int16))
    B = dev(WL.bf16_bits(B0).view(np.int16))
    state = dict(A32=dev(A0), B32=dev(B0), mA=t.zeros((m, r), device="cuda"), vA=t.zeros((m, r), device="cuda"),
                 mB=t.zeros((r, k), device="cuda"), vB=t.zeros((r, k), device="cuda"),
                 ms=t.zeros(s_shape, device="cuda"), vs=t.zeros(s_shape, device="cuda"))
    s = dev(s0)
    ref = {"A": (A0.astype(np.float64), np.zeros((m, r)), np.zeros((m, r))),
           "B": (B0.astype(np.float64), np.zeros((r, k)), np.zeros((r, k))),
           "s": (s0.astype(np.float64), np.zeros(s_shape), np.zeros(s_shape))}
    lrs = {"A": 1e-3, "B": 1e-3, "s": 1e-4}
    sqn = t.zeros((1,), dtype=t.float32, device="cuda")
    for step in range(1, 4):
        scale = 5.0 if step == 2 else 0.001           # step 2 clips, the others do not
        grads = {"A": rng.standard_normal((m, r)) * scale, "B": rng.standard_normal((r, k)) * scale,
                 "s": rng.standard_normal(s_shape) * scale}
        g32 = {n: g.astype(np.float32) for n, g in grads.items()}
        # a second, smaller layer whose gradients also enter the global norm
        o32 = [(rng.standard_normal(sh) * scale).astype(np.float32) for sh in ((128, 8), (8, 128), (128,))]
        sqn.zero_()
        LQ.grad_sqnorm(L, dev(g32["A"]), dev(g32["B"]), dev(g32["s"]), sqn)
        LQ.grad_sqnorm(L_other, *[dev(o) for o in o32], sqn)
        allg = [g32["A"], g32["B"], g32["s"]] + o32
        coef = O.clip_coefficient(allg, 1.0)
        total = sum(float(np.sum(g.astype(np.float64) ** 2)) for g in allg)
        assert abs(float(sqn.item()) - total) <= 1e-5 * total
        opt = LQ.AdamW.make(lrs["A"], lrs["s"], step=step)
        LQ.adamw_step(L, opt, sqn, dev(g32["A"]), dev(g32["B"]), dev(g32["s"]), state, s, A, B)
        for n in ("A", "B", "s"):
            ref[n] = O.adamw_update(ref[n][0], coef * g32[n].astype(np.float64), ref[n][1], ref[n][2], step, lrs[n])
    LQ.get_device_status()
    for n, got in (("A", state["A32"]), ("B", state["B32"]), ("s", s)):
        np.testing.assert_allclose(got.cpu().numpy().astype(np.float64), ref[n][0], rtol=2e-5, atol=1e-7, err_msg=n)
    for n, mm, vv in (("A", "mA", "vA"), ("B", "mB", "vB"), ("s", "ms", "vs")):
        np.testing.assert_allclose(state[mm].cpu().numpy(), ref[n][1], rtol=1e-4, atol=1e-9, err_msg=mm)
        np.testing.assert_allclose(state[vv].cpu().numpy(), ref[n][2], rtol=1e-4, atol=1e-12, err_msg=vv)
    # the bf16 copies are the round-to-nearest-even images of the fp32 masters
    np.testing.assert_array_equal(A.cpu().numpy().view(np.uint16), WL.bf16_bits(state["A32"].cpu().numpy()))
    np.testing.assert_array_equal(B.cpu().numpy().view(np.uint16), WL.bf16_bits(state["B32"].cpu().numpy()))
