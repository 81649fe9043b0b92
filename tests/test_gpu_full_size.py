"""GPU parity at the benchmark's full sizes, in the launch configuration that
bench.py times: one lrqat_linear_fwd and one lrqat_linear_bwd call over all
T tokens of a LLaMA-shaped layer (T = 16384 for the three projection shapes of
the LLaMA-2-13B decoder layer, 8192 for the others).

The oracle cannot redo a full 8192-token layer in a test's time, so it checks
what it can compute exactly, one piece at a time:
  * every integer code of W_hat that the fused producers build, bit for bit
    (identity inputs turn the forward output into C^T and the dX output into C;
    near-ties exempt, as in the small-size tests);
  * Y and dX at sampled token rows (all output columns of those rows);
  * dA and ds at sampled weight rows and dB at sampled weight columns, from the
    rows / columns of G = dY^T X_hat that the oracle forms in fp64;
  * every code of W_Z from lrqat_merge at the largest merged projection.
Sampled outputs are compared with the same relative Frobenius tolerances as the
small-size tests (1e-2 for Y and dX, 2e-2 for the adapter and scale gradients).

Every case reports what it found, pass or fail: the number of codes checked, the
near-tie exemptions and mismatches, and the five relative errors, as one JSON line
on stdout (shown by `pytest -rA`) and, when LRQAT_PARITY_REPORT names a file,
appended to it.
"""
import dataclasses
import json
import os

import numpy as np
import pytest

import oracle as O
from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL

from gpu_util import DeviceLayer, bits_to_f32, oracle_layer, to_dev, torch

pytestmark = pytest.mark.gpu

TOL_ACT = 1e-2
TOL_GRAD = 2e-2

# The three projection shapes of the LLaMA-2-13B decoder layer that bench.py times by
# default (q/k/v/o 5120 x 5120, gate/up 13824 x 5120, down 5120 x 13824; T = 16384), the
# 4096 x 4096 layer (Q4.4 per channel), the largest projection of the W4 g128 + A8 MLP
# (14336 x 4096), the INT-3 packed down projection (4096 x 11008), and the 4096 x 4096
# layer with asymmetric W2, per-token A8, and BF16 / FP8 bases (T = 8192).
_L13 = WL.workload("llama2_13b_layer")
FULL_CASES = [
    ("llama2_13b_qkvo", _L13.layers[0], _L13.tokens),
    ("llama2_13b_gate", _L13.layers[4], _L13.tokens),
    ("llama2_13b_down", _L13.layers[6], _L13.tokens),
    ("llama2_7b_attn", WL.workload("llama2_7b_attn").layers[0], 8192),
    ("llama3_8b_gate_g128_a8", WL.workload("llama3_8b_mlp").layers[0], 8192),
    ("llama2_7b_down_int3", WL.workload("llama2_7b_mlp").layers[2], 8192),
    ("llama2_7b_attn_int2_asym", WL.workload("llama2_7b_attn_int2").layers[0], 8192),
    ("llama2_7b_attn_w4a8_token", WL.workload("llama2_7b_attn_w4a8").layers[0], 8192),
    ("llama2_7b_attn_phi_bf16", WL.workload("llama2_7b_attn_phi_bf16").layers[0], 8192),
    ("llama2_7b_attn_phi_fp8", WL.workload("llama2_7b_attn_phi_fp8").layers[0], 8192),
    ("llama2_7b_attn_r256", WL.workload("llama2_7b_attn_r256").layers[0], 8192),
]


# The source of the GEMMs' low-rank term (lrqat_set_lowrank_path): at these token counts the
# default takes the codes pass; the 13B q/k/v/o shape and the 4096 x 4096 layer also run with
# the tile each GEMM stage computes.
_BOTH_PATHS = ("llama2_13b_qkvo", "llama2_7b_attn")
FULL_PATH_CASES = [pytest.param(*c, p, id=f"{c[0]}-{p}") for c in FULL_CASES
                   for p in (("tile", "codes") if c[0] in _BOTH_PATHS else ("auto",))]


def _report(test: str, cid: str, **fields):
    """One JSON line per case: on stdout and, with LRQAT_PARITY_REPORT set, in that file."""
    line = json.dumps(dict(test=test, case=cid, **fields), sort_keys=True)
    print(line)
    path = os.environ.get("LRQAT_PARITY_REPORT")
    if path:
        with open(path, "a") as f:
            f.write(line + "\n")


def _oracle_base(data, OL):
    """The oracle's range setting and downcast: (s0, z0 or None, Phi0)."""
    if data.spec.asym:
        s0, z0 = O.minmax_range_asym(data.W0, OL)
        return s0, z0, O.downcast(data.W0, s0, OL, z0)
    s0 = O.minmax_scale(data.W0, OL)
    return s0, None, O.downcast(data.W0, s0, OL)


def _codes_spec(spec):
    # the codes do not depend on the activation quantizer; identity inputs need it off
    return WL.LayerSpec(spec.name, spec.m, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format,
                        0, spec.w_std, spec.outlier_frac, spec.outlier_mult, spec.a_std, spec.b_std, spec.asym,
                        spec.w_row_shift, False)


@pytest.mark.parametrize("cid,spec,T,path", FULL_PATH_CASES)
def test_full_size_codes_bit_exact(cid, spec, T, path, lowrank_path):
    lowrank_path(path)
    t = torch()
    spec = _codes_spec(spec)
    data = WL.make_layer(spec, 1, seed=3, with_activations=False)
    dl = DeviceLayer(data)
    dl.s = t.ones_like(dl.s)
    L = dl.layer
    m, k = spec.m, spec.k
    # forward with X = I_k: Y[j, i] = c[i, j]
    X = t.eye(k, dtype=t.bfloat16, device="cuda").view(t.int16)
    Y = t.empty((k, m), dtype=t.int16, device="cuda")
    ws = t.empty(max(LQ.fwd_workspace_bytes(L, k), 16), dtype=t.uint8, device="cuda")
    LQ.linear_fwd(L, k, X, dl.phi0, dl.s, dl.A, dl.B, None, Y, ws)
    c_fwd = bits_to_f32(Y).T
    del X, Y, ws
    # dX with dY = I_m: dX[i, j] = c[i, j]
    dYe = t.eye(m, dtype=t.bfloat16, device="cuda").view(t.int16)
    Xz = t.zeros((m, k), dtype=t.int16, device="cuda")
    dX = t.empty((m, k), dtype=t.int16, device="cuda")
    dA = t.empty((m, spec.r), dtype=t.float32, device="cuda")
    dB = t.empty((spec.r, k), dtype=t.float32, device="cuda")
    ds = t.empty_like(dl.s)
    wsb = t.empty(LQ.bwd_workspace_bytes(L, m), dtype=t.uint8, device="cuda")
    LQ.linear_bwd(L, m, dYe, Xz, dl.phi0, dl.s, dl.A, dl.B, None, dX, dA, dB, ds, False, wsb)
    LQ.get_device_status()
    c_dx = bits_to_f32(dX)
    OL = oracle_layer(spec)
    _, z0, phi0 = _oracle_base(data, OL)
    u = O.preround(phi0, data.A, data.B, OL)
    c = O.codes_from_u(u, OL)[1] - O.expand_zero(z0, OL)   # the operand holds c - z
    exempt = O.near_tie(u)
    bad = {name: int(((got != c) & ~exempt).sum()) for name, got in (("fwd", c_fwd), ("dX", c_dx))}
    _report("codes", cid, path=LQ.lowrank_path(), codes=int(c.size), near_tie_exempt=int(exempt.sum()), mismatches_fwd=bad["fwd"],
            mismatches_dx=bad["dX"], differ_at_exempt=int(((c_fwd != c) & exempt).sum()))
    for name, n in bad.items():
        assert n == 0, f"{name}: {n} code mismatches of {c.size} (near-ties exempt: {exempt.sum()})"


@pytest.mark.parametrize("cid,spec,T,path", FULL_PATH_CASES)
def test_full_size_sampled_outputs(cid, spec, T, path, lowrank_path):
    lowrank_path(path)
    t = torch()
    data = WL.make_layer(spec, T, seed=11)
    dl = DeviceLayer(data)
    L = dl.layer
    X, dY = to_dev(data.X_bits), to_dev(data.dY_bits)
    s_x_host, s_x = None, None
    if spec.act_bits == 8 and not spec.act_per_token:
        s_x_host = np.float32(np.float32(np.abs(data.X).max()) / np.float32(127.0))
        s_x = t.tensor([s_x_host], dtype=t.float32, device="cuda")
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

    OL = oracle_layer(spec)
    s0, z0, phi0 = _oracle_base(data, OL)
    fq = O.fake_quant_weight(phi0, s0, data.A, data.B, OL, z0)
    if spec.act_bits == 8 and spec.act_per_token:
        _, Xh, Mx, _ = O.act_quant_per_token(data.X)
    elif spec.act_bits == 8:
        _, Xh, Mx = O.act_quant(data.X, s_x_host)
    else:
        Xh = data.X.astype(np.float64)
        Mx = np.ones_like(Xh)
    dYf = data.dY.astype(np.float64)
    scale = OL.alpha / OL.r

    # Y and dX at sampled token rows (every column)
    ts = WL.token_sample(T, 24, seed=1)
    Y_ref = Xh[ts] @ fq["W_hat"].T
    dX_ref = (dYf[ts] @ fq["W_hat"]) * Mx[ts]
    Y_got = bits_to_f32(Y[t.as_tensor(ts, device="cuda")])
    dX_got = bits_to_f32(dX[t.as_tensor(ts, device="cuda")])
    errs = {"Y": O.rel_fro(Y_got, Y_ref), "dX": O.rel_fro(dX_got, dX_ref)}

    # dA and ds at sampled weight rows: rows of G, dU and the codes
    rows = WL.token_sample(spec.m, 6, seed=2)
    G_rows = dYf[:, rows].T @ Xh
    s_rows = O.expand_scale(s0, OL)[rows]
    dU_rows = G_rows * s_rows * fq["M"][rows]
    dA_ref = scale * (dU_rows @ data.B.astype(np.float64).T)
    Gc = G_rows * fq["cz"][rows]
    ds_ref = Gc.sum(axis=1) if spec.group_size == 0 else Gc.reshape(len(rows), -1, spec.group_size).sum(axis=2)
    dA_got = dA.cpu().numpy()[rows]
    ds_got = ds.cpu().numpy().reshape((spec.m, -1) if spec.group_size else (spec.m,))[rows]
    errs["dA"] = O.rel_fro(dA_got, dA_ref)
    errs["ds"] = O.rel_fro(ds_got, ds_ref)

    # dB at sampled weight columns: columns of G and dU
    cols = WL.token_sample(spec.k, 6, seed=3)
    G_cols = dYf.T @ Xh[:, cols]
    dU_cols = G_cols * O.expand_scale(s0, OL)[:, cols] * fq["M"][:, cols]
    dB_ref = scale * (data.A.astype(np.float64).T @ dU_cols)
    dB_got = dB.cpu().numpy()[:, cols]
    errs["dB"] = O.rel_fro(dB_got, dB_ref)
    _report("sampled_outputs", cid, path=LQ.lowrank_path(), T=T, rel_err=errs, token_rows=len(ts), weight_rows=len(rows),
            weight_cols=len(cols))
    for key in ("Y", "dX"):
        assert errs[key] <= TOL_ACT, errs
    for key in ("dA", "dB", "ds"):
        assert errs[key] <= TOL_GRAD, errs


# The merge of the largest projection of the 13B layer that bench.py times with merge
# (the 5120 x 13824 down projection), plus the 4096 x 4096 layer with a
# rank that is not a multiple of 8 (the CUDA-core merge) and with a BF16 base.  The
# factors are drawn large enough (|A B| ~ 0.5 code steps) that many codes move away from
# the base's.
def _merge_spec(spec):
    return dataclasses.replace(spec, a_std=0.25, b_std=0.25)


MERGE_CASES = [
    ("llama2_13b_down", _merge_spec(WL.workload("llama2_13b_layer").layers[6])),
    ("llama2_7b_attn_r20", WL.LayerSpec("attn_r20", 4096, 4096, 20, 20.0, 4, 0, WL.PHI_QFIXED, a_std=0.25,
                                        b_std=0.25)),
    ("llama2_7b_attn_phi_bf16", _merge_spec(WL.workload("llama2_7b_attn_phi_bf16").layers[0])),
    ("llama2_7b_attn_r256", dataclasses.replace(WL.workload("llama2_7b_attn_r256").layers[0], a_std=0.15,
                                                b_std=0.15)),
]


@pytest.mark.parametrize("cid,spec", MERGE_CASES, ids=[c[0] for c in MERGE_CASES])
def test_full_size_merge_bit_exact(cid, spec):
    """Every code of W_Z from lrqat_merge against the oracle's merge (near-ties exempt)."""
    t = torch()
    data = WL.make_layer(spec, 1, seed=5, with_activations=False)
    dl = DeviceLayer(data)
    wz = t.empty((spec.m, spec.k), dtype=t.int8, device="cuda")
    LQ.merge(dl.layer, dl.phi0, dl.A, dl.B, wz)
    LQ.get_device_status()
    got = wz.cpu().numpy()
    OL = oracle_layer(spec)
    _, _, phi0 = _oracle_base(data, OL)
    ref = O.merge(phi0, data.A, data.B, OL)
    exempt = O.near_tie(O.preround(phi0, data.A, data.B, OL))
    bad = (got != ref) & ~exempt
    _report("merge", cid, codes=int(ref.size), near_tie_exempt=int(exempt.sum()), mismatches=int(bad.sum()),
            differ_at_exempt=int(((got != ref) & exempt).sum()))
    assert bad.sum() == 0, f"{bad.sum()} code mismatches of {ref.size} (near-ties exempt: {exempt.sum()})"
    assert (ref != O.merge(phi0, data.A, np.zeros_like(data.B), OL)).mean() > 0.1   # the low-rank term matters
