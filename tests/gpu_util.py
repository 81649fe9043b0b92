"""Helpers for the GPU parity tests: host arrays <-> device tensors, and the
per-layer set-up that goes through the library's own entry points."""
import numpy as np

from paper_2406_06385_gb300 import lrqat as LQ
from paper_2406_06385_gb300 import workloads as WL


def torch():
    import torch as _t
    return _t


def to_dev(a: np.ndarray):
    t = torch()
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return t.from_numpy(a.view(np.int16)).cuda()
    if a.dtype == np.uint8:
        return t.from_numpy(a).cuda()
    return t.from_numpy(a).cuda()


def bits_to_f32(t) -> np.ndarray:
    """Device bf16 bits (int16 tensor) -> host fp32 values."""
    return WL.bf16_to_f32(t.cpu().numpy().view(np.uint16))


def empty(shape, dtype):
    t = torch()
    return t.empty(shape, dtype=dtype, device="cuda")


def oracle_layer(spec):
    import oracle as O
    return O.Layer(spec.m, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format, spec.act_bits,
                   spec.act_per_token, spec.u_bf16)


PHI_HOST_DTYPE = {WL.PHI_QFIXED: np.int8, WL.PHI_INT_PACKED: np.uint8, WL.PHI_BF16: np.uint16,
                  WL.PHI_FP16: np.uint16, WL.PHI_FP8_E4M3: np.uint8, WL.PHI_FP8_E5M2: np.uint8}


def phi_buffer(spec):
    """Device buffer of Phi0 in the layer's storage format (see lrqat_phi_format)."""
    t = torch()
    if spec.phi_format == WL.PHI_INT_PACKED:
        return t.empty((spec.m, spec.k // 2), dtype=t.uint8, device="cuda")
    if spec.phi_format in (WL.PHI_BF16, WL.PHI_FP16):
        return t.empty((spec.m, spec.k), dtype=t.int16, device="cuda")
    return t.empty((spec.m, spec.k), dtype=t.int8 if spec.phi_format == WL.PHI_QFIXED else t.uint8, device="cuda")


def near_bf16_boundary(A, B, rel: float = 2.0 ** -18) -> np.ndarray:
    """Elements whose exact A B lies so close to a bf16 rounding boundary that the
    fp32-accumulated product of the tensor cores may round to the other neighbour
    (the bf16 pre-round reading rounds A B to bf16 first)."""
    import oracle as O
    ab = np.asarray(A, dtype=np.float64) @ np.asarray(B, dtype=np.float64)
    return O.bf16_round(ab * (1 + rel)) != O.bf16_round(ab * (1 - rel))


def phi_host(phi0, spec) -> np.ndarray:
    """Device Phi0 -> host array in the oracle's representation of the format."""
    return phi0.cpu().numpy().view(PHI_HOST_DTYPE[spec.phi_format])


class DeviceLayer:
    """One layer's frozen base and adapters on the device, prepared with the
    library's own range setting and downcast."""

    def __init__(self, data: WL.LayerData, s_scale: float = 1.0):
        t = torch()
        spec = data.spec
        self.spec = spec
        self.W0 = to_dev(data.W0)
        ng = spec.k // spec.group_size if spec.group_size else 1
        self.s0 = t.empty((spec.m, ng) if spec.group_size else (spec.m,), dtype=t.float32, device="cuda")
        # asymmetric weights: the range setting writes the zero offsets, later calls read them
        self.z = t.empty_like(self.s0) if spec.asym else None
        self.layer = LQ.Layer.from_spec(spec, self.z.data_ptr() if spec.asym else 0)
        LQ.range_minmax(self.layer, self.W0, self.s0)
        self.phi0 = phi_buffer(spec)
        LQ.downcast(self.layer, self.W0, self.s0, self.phi0)
        self.s = (self.s0 * s_scale).contiguous()
        self.A = to_dev(data.A_bits)
        self.B = to_dev(data.B_bits)
