"""The C-ABI library loads, exports every symbol include/lrqat.h declares, and
rejects bad arguments on the host before any CUDA work (no GPU needed)."""
import ctypes
import os
import re

import pytest

from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300.build import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build()
    return LQ.lib()


def header_functions():
    src = open(os.path.join(ROOT, "include", "lrqat.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\*?\s+\**(lrqat_[a-z_0-9]+)\s*\(", src, flags=re.M)))


def test_header_declares_the_entry_points():
    names = header_functions()
    for expected in ("lrqat_range_minmax", "lrqat_downcast", "lrqat_linear_fwd", "lrqat_linear_bwd", "lrqat_merge",
                     "lrqat_fwd_workspace_bytes", "lrqat_bwd_workspace_bytes", "lrqat_get_device_status",
                     "lrqat_last_error", "lrqat_grad_sqnorm", "lrqat_adamw_step", "lrqat_range_lp", "lrqat_act_quant"):
        assert expected in names


def test_library_exports_every_declared_symbol(lib):
    for name in header_functions():
        assert hasattr(lib, name), name


def _layer(**kw):
    d = dict(m=256, k=256, r=4, alpha=4.0, bits=4, group_size=0, phi_format=LQ.PHI_QFIXED, act_bits=0)
    d.update(kw)
    return LQ.Layer(**d)


@pytest.mark.parametrize("kw,status", [
    (dict(m=100), -2), (dict(k=0), -1), (dict(r=0), -1), (dict(r=257), -2), (dict(bits=1), -1), (dict(bits=8), -1),
    (dict(r=65, bits=8, phi_format=LQ.PHI_BF16), -2),
    (dict(phi_format=LQ.PHI_INT_PACKED, bits=5), -1), (dict(group_size=64), -2), (dict(group_size=384), -2),
    (dict(act_bits=4), -2), (dict(phi_format=7), -1),
])
def test_invalid_layers_are_rejected_on_host(lib, kw, status):
    L = _layer(**kw)
    got = lib.lrqat_linear_fwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, None, 16, 16, 1 << 20, None)
    assert got == status, LQ.last_error()
    assert LQ.last_error()


def test_null_and_misaligned_pointers_are_rejected(lib):
    L = _layer()
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 64, None, 16, 16, 16, 16, None, 16, 16, 1 << 20, None) == -1
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 64, 18, 16, 16, 16, 16, None, 16, 16, 1 << 20, None) == -3
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 0, 16, 16, 16, 16, 16, None, 16, 16, 1 << 20, None) == -1
    # act_bits = 8 needs s_x
    L8 = _layer(act_bits=8)
    assert lib.lrqat_linear_fwd(ctypes.byref(L8), 64, 16, 16, 16, 16, 16, None, 16, 16, 1 << 30, None) == -1


def test_short_workspace_is_rejected(lib):
    L = _layer()
    need = lib.lrqat_fwd_workspace_bytes(ctypes.byref(L), 64)
    assert need > 0
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, None, 16, 16, need - 1, None) == -4
    assert lib.lrqat_linear_bwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, 16, None, 16, 16, 16, 16, 0, None, 0,
                                None) in (-4, -5)   # -5 when no CUDA device is visible


def test_workspace_grows_with_tokens_and_activation_quantizer(lib):
    L = _layer()
    L8 = _layer(act_bits=8)
    assert lib.lrqat_fwd_workspace_bytes(ctypes.byref(L), 64) == lib.lrqat_fwd_workspace_bytes(ctypes.byref(L), 4096)
    assert lib.lrqat_fwd_workspace_bytes(ctypes.byref(L8), 4096) >= 4096 * 256 * 2
    assert lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), 64) > 0
    assert lib.lrqat_fwd_workspace_bytes(ctypes.byref(_layer(m=100)), 64) == 0


def test_group_wise_forward_workspace_holds_the_scale_rows(lib):
    """A group-wise forward stages its scales (and zero offsets) as bf16 rows [groups][m], so
    its workspace covers groups x m x 2 bytes per array beyond the per-channel layer's."""
    m, k, g = 512, 1024, 128
    pc = lib.lrqat_fwd_workspace_bytes(ctypes.byref(_layer(m=m, k=k)), 64)
    gw = lib.lrqat_fwd_workspace_bytes(ctypes.byref(_layer(m=m, k=k, group_size=g)), 64)
    gz = lib.lrqat_fwd_workspace_bytes(ctypes.byref(_layer(m=m, k=k, group_size=g, zero=256)), 64)
    assert gw - pc >= (k // g) * m * 2
    assert gz - gw >= (k // g) * m * 2


def test_quantizer_setting_fields_are_checked_on_host(lib):
    """act_per_token needs act_bits 8; the zero offsets must be 16-byte aligned."""
    L = _layer(act_per_token=1)
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, None, 16, 16, 1 << 20, None) == -1
    L = _layer(zero=8)
    assert lib.lrqat_linear_fwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, None, 16, 16, 1 << 20, None) == -3


def test_adamw_arguments_are_checked_on_host(lib):
    L = _layer()
    st = LQ.AdamWState(*([16] * 8))
    ok = LQ.AdamW.make(1e-3, 0.0, step=1)
    args = lambda opt, state: (ctypes.byref(L), ctypes.byref(opt), 16, 16, 16, 16, state, 16, 16, 16, None)
    assert lib.lrqat_adamw_step(*args(LQ.AdamW.make(1e-3, 0.0, step=0), ctypes.byref(st))) == -1
    assert lib.lrqat_adamw_step(*args(LQ.AdamW.make(1e-3, 0.0, step=1, beta2=1.0), ctypes.byref(st))) == -1
    assert lib.lrqat_adamw_step(*args(ok, None)) == -1
    assert lib.lrqat_grad_sqnorm(ctypes.byref(L), None, 16, 16, 16, None) == -1


def test_lp_range_arguments_are_checked_on_host(lib):
    L = _layer()
    f = lib.lrqat_range_lp
    assert f(ctypes.byref(L), 16, 0.0, 100, 16, None) == -1
    assert f(ctypes.byref(L), 16, float("nan"), 100, 16, None) == -1
    assert f(ctypes.byref(L), 16, 2.0, 0, 16, None) == -1
    assert f(ctypes.byref(L), 16, 2.0, 257, 16, None) == -1
    assert f(ctypes.byref(L), None, 2.0, 100, 16, None) == -1
    assert f(ctypes.byref(_layer(zero=16)), 16, 2.0, 100, 16, None) == -2
    assert f(ctypes.byref(_layer(k=65536)), 16, 2.0, 100, 16, None) == -2


def test_bf16_pre_round_is_checked_on_host(lib):
    f = lambda L: lib.lrqat_linear_fwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, None, 16, 16, 1 << 20, None)
    assert f(_layer(u_bf16=2)) == -1
    assert f(_layer(u_bf16=1, phi_format=LQ.PHI_FP16)) == -2
    assert f(_layer(u_bf16=1, alpha=3.0)) == -2            # alpha / r = 3/4: not a power of two
    assert f(_layer(u_bf16=1, zero=16)) == -2


def test_act_quant_arguments_are_checked_on_host(lib):
    f = lib.lrqat_act_quant
    assert f(ctypes.byref(_layer()), 64, 16, 16, 16, None, None) == -1                 # act_bits 0
    assert f(ctypes.byref(_layer(act_bits=8)), 64, 16, None, 16, None, None) == -1     # per tensor needs s_x
    assert f(ctypes.byref(_layer(act_bits=8)), 0, 16, 16, 16, None, None) == -1
    assert f(ctypes.byref(_layer(act_bits=8)), 64, 16, 16, 18, None, None) == -3
    assert f(ctypes.byref(_layer(act_bits=8)), 64, 16, 16, 16, 18, None) == -3


def test_quantized_activation_entry_points_are_checked_on_host(lib):
    fq, bq = lib.lrqat_linear_fwd_quantized, lib.lrqat_linear_bwd_quantized
    a8, a8t = _layer(act_bits=8), _layer(act_bits=8, act_per_token=1)
    assert fq(ctypes.byref(_layer()), 64, 16, 16, 16, 16, 16, 16, 16, 16, 1 << 20, None) == -1   # act_bits 0
    bwd = lambda L, mask: bq(ctypes.byref(L), 64, 16, 16, mask, 16, 16, 16, 16, 16, 16, 16, 16, 16, 0, 16, 1 << 20,
                             None)
    assert bwd(_layer(), 16) == -1                 # act_bits 0
    assert bwd(a8, None) == -1                     # per tensor needs the clip mask
    assert bwd(a8, 18) == -3                       # mask not 4-byte aligned
    assert bwd(a8t, 18) == -3
    assert "mask" in LQ.last_error()


def test_dw_schedule_choice_of_the_cost_model(lib, dw_schedule):
    """The plan without an override (152 SMs assumed when no GPU is present):
      - 4096 x 4096 at 8192 tokens, 512 tiles: whole-tile waves (3 x 152) and the 56 remaining
        tiles cut into 2 or 3 token parts, one per CTA, beat two equal token splits per tile
        (3 partial slots per tile against 2);
      - 2432 x 2048 at 8192 tokens, exactly 152 tiles: one wave of whole tiles, no tail, so equal
        splits are taken and the tail override cannot apply;
      - 384 x 512 at 1000 tokens, 6 tiles: 8 parts a tile keep 48 SMs busy with 4 stages each,
        against 24 SMs with 8 stages each, so the tail schedule is taken (8 slots against 4).
    The backward workspace sizes (the partial slots) show which plan was made."""
    cases = {"big": (_layer(m=4096, k=4096, r=32, alpha=32.0), 8192),
             "waves": (_layer(m=2432, k=2048, r=32, alpha=32.0), 8192),
             "tiny": (_layer(m=384, k=512, r=32, alpha=32.0), 1000)}
    sizes = {}
    for sched in ("auto", "split", "tail"):
        dw_schedule(sched)
        sizes[sched] = {n: lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), T) for n, (L, T) in cases.items()}
    assert sizes["auto"]["big"] == sizes["tail"]["big"] > sizes["split"]["big"]
    assert sizes["auto"]["waves"] == sizes["split"]["waves"] == sizes["tail"]["waves"]
    assert sizes["auto"]["tiny"] == sizes["tail"]["tiny"] > sizes["split"]["tiny"]
    assert lib.lrqat_set_dw_schedule(3) == -1 and lib.lrqat_set_dw_schedule(-1) == -1


def test_dw_schedule_environment_is_read_once_at_load(lib, dw_schedule, monkeypatch):
    """LRQAT_DW_SCHEDULE sets the start value when the library is loaded; changing the
    environment afterwards changes no workspace size (so a size query and the call that
    uses it always agree)."""
    L = _layer(m=4096, k=4096, r=32, alpha=32.0)
    dw_schedule("auto")
    before = lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), 8192)
    monkeypatch.setenv("LRQAT_DW_SCHEDULE", "split")
    assert lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), 8192) == before
    dw_schedule("split")
    split = lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), 8192)
    assert split < before
    # a fresh process that loads the library with the variable set starts from it
    code = ("import ctypes, sys; sys.path.insert(0, %r); from paper_2406_06385_gb300 import lrqat as LQ; "
            "L = LQ.Layer(4096, 4096, 32, 32.0, 4, 0, 0, 0); "
            "print(LQ.lib().lrqat_bwd_workspace_bytes(ctypes.byref(L), 8192))" % ROOT)
    import subprocess
    import sys
    env = dict(os.environ, LRQAT_DW_SCHEDULE="split")
    out = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stderr
    assert int(out.stdout.strip()) == split


def test_lowrank_path_setting(lib, lowrank_path, monkeypatch):
    """The source of the GEMMs' low-rank term is a process-wide setting whose start value
    comes from LRQAT_LOWRANK_PATH at load; the workspace sizes cover every setting (so a size
    query and the call that uses it agree whatever the setting is), and the forward's size holds
    the m x k int8 codes of the weights."""
    L = _layer(m=4096, k=4096, r=32, alpha=32.0)
    sizes = {}
    for path in ("auto", "tile", "codes"):
        lowrank_path(path)
        assert LQ.lowrank_path() == path
        sizes[path] = (lib.lrqat_fwd_workspace_bytes(ctypes.byref(L), 8192),
                       lib.lrqat_bwd_workspace_bytes(ctypes.byref(L), 8192))
    assert sizes["auto"] == sizes["tile"] == sizes["codes"]
    assert sizes["auto"][0] >= 4096 * 4096 and sizes["auto"][1] >= 2 * 4096 * 4096
    assert lib.lrqat_set_lowrank_path(3) == -1 and lib.lrqat_set_lowrank_path(-1) == -1
    code = ("import sys; sys.path.insert(0, %r); from paper_2406_06385_gb300 import lrqat as LQ; "
            "print(LQ.lowrank_path())" % ROOT)
    import subprocess
    import sys
    for value, expect in (("tile", "tile"), ("codes", "codes"), ("bogus", "auto")):
        env = dict(os.environ, LRQAT_LOWRANK_PATH=value)
        out = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=120)
        assert out.returncode == 0, out.stderr
        assert out.stdout.strip() == expect


def test_gradient_outputs_must_be_16_byte_aligned(lib):
    """The gradient reduction reads and writes dA and dB with 16-byte accesses, so an
    unaligned dA or dB is rejected on the host before any launch (ds may be unaligned)."""
    L = _layer()
    f = lambda dA, dB, ds: lib.lrqat_linear_bwd(ctypes.byref(L), 64, 16, 16, 16, 16, 16, 16, None, 16, dA, dB, ds, 0,
                                                16, 1 << 30, None)
    assert f(20, 16, 16) == -3 and "dA" in LQ.last_error()
    assert f(16, 20, 16) == -3 and "dB" in LQ.last_error()
    assert f(16, 16, None) == -1
    assert f(None, 16, 16) == -1
