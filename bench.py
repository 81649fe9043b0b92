"""Throughput benchmark of the GB300 LR-QAT linear layer (fwd + bwd).

One step = LR-QAT forward and backward of every layer of the workload over one
batch of T tokens, with the fake-quantized weight rebuilt on chip in each of the
three GEMMs (Eq. 8 of the paper, checkpointed as in Sec. 3).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...     # the CPU oracle, timed on host cores

Prints ONE JSON line (rank 0).  With N > 1 (torchrun) every rank runs an
independent replica of the workload (weak scaling, no collective on the data
path); the timed region is bracketed by a barrier and device synchronization,
and the slowest rank's time is used.  The device-resident timed region replays
each step's library calls from CUDA graphs captured once per input set (the same
kernels; --no-graph times the eager calls); the end-to-end figure (host buffers,
copies included) and the per-kernel traced pass use eager calls.
"""
from __future__ import annotations

import argparse
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time
import hashlib

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "LR-QAT linear fwd+bwd tokens/s and TFLOP/s, fraction of GB300 bf16 dense peak"
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
GEMM_KERNELS = ("fused_fwd", "fused_dx", "fused_dw")
# the sources whose kernels a traced name can refer to (the forward and dX run on CTA pairs or on one SM)
KERNEL_SOURCES = {"fused_fwd": ("fused_gemm.cu", "fused_pair.cu"), "fused_dx": ("fused_gemm.cu", "fused_pair.cu"),
                  "fused_dw": ("dw.cu", "dw_pair.cu")}


# --------------------------------------------------------------------------- helpers

def phi_label(fmt: int, bits: int) -> str:
    """Storage format of Phi0 (the lrqat_phi_format values) as a config label."""
    return {0: "Q%d.%d int8" % (bits, 8 - bits), 1: f"INT-{bits} packed", 2: "BF16", 3: "FP16", 4: "FP8 E4M3",
            5: "FP8 E5M2"}[fmt]

def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {k: float(p[k]) for k in FALLBACK_PEAKS}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def kernel_source_hash(kernel: str) -> str:
    """sha256 of the sources that define a kernel (its .cu file and the shared device headers)."""
    csrc = os.path.join(ROOT, "paper_2406_06385_gb300", "csrc")
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel] + ("ptx.cuh", "quant.cuh", "kernels.h"):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary of this kernel and workload,
    or None when there is none or the kernel's source changed since it was captured."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    mb = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    ms = re.search(r"source_sha256_16:\s*([0-9a-f]+)", text)
    if not mb or not ms or ms.group(1) != kernel_source_hash(kernel):
        return None
    return float(mb.group(1))


def peak_kind(clk) -> str:
    """"sustained" when the clock record of the timed region shows the power cap or a median
    SM clock below 97% of the maximum, else "burst"."""
    if "sw_power_cap" in (clk.get("reasons") or []):
        return "sustained"
    sm, smax = clk.get("sm_mhz"), clk.get("sm_max_mhz")
    if sm is not None and smax and sm < 0.97 * smax:
        return "sustained"
    return "burst"


def kernel_bytes(T: int, spec) -> float:
    """Algorithmic HBM bytes of one launch of any of the three GEMM kernels: two bf16 token
    operands of T rows (forward: X [T, k] in, Y [T, m] out; dX: dY [T, m] in, dX [T, k]
    out; dW: dY and X in), the stored base once and the bf16 adapters.  The dW kernel's
    per-tile gradient partials are not counted (their size depends on the schedule)."""
    base = spec.m * spec.k * (0.5 if spec.phi_format == 1 else 2.0 if spec.phi_format in (2, 3) else 1.0)
    return 2.0 * T * (spec.m + spec.k) + base + 2.0 * spec.r * (spec.m + spec.k)


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons every 200 ms while running."""

    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="lrqat_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.out, stderr=subprocess.DEVNULL)
            time.sleep(0.6)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.out.close()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 11:
                    continue
                rows.append(parts)
        except OSError:
            pass
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        mine = [r for r in rows if self.uuid and r[1] == self.uuid]
        rows = mine or [r for r in rows if r[0] == rows[0][0]] if rows else rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        busy = [r for r in rows if _num(r[5]) is not None and _num(r[5]) >= 50] or rows
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in busy for n, v in zip(names, r[7:11]) if v.lower().startswith("active")})
        sm = [_num(r[2]) for r in busy if _num(r[2]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": _num(busy[0][3]),
                "power_w_max": max((_num(r[4]) or 0.0) for r in busy), "reasons": reasons, "samples": len(busy)}


def _num(s):
    try:
        return float(s)
    except (TypeError, ValueError):
        return None


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), int(os.environ.get("LOCAL_RANK", "0"))


def aggregate_over_ranks(ms: float, units: float):
    """Slowest rank's time and the sum of units over ranks (no-op without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return ms, units
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def workload_config(wl, args, world: int) -> dict:
    """The `config` object of the JSON line: the workload by name, its layer shapes and
    quantizer settings, and how the timed region launches and rotates its inputs.  Both
    arms print the same object for the same arguments."""
    spec0 = wl.layers[0]
    in_bytes = args.sets * sum(2 * wl.tokens * (l.k + l.m) for l in wl.layers)
    return {"workload": wl.name, "tokens": wl.tokens, "layers": [f"{l.name}:{l.m}x{l.k}" for l in wl.layers],
            "r": spec0.r, "alpha": spec0.alpha, "bits": spec0.bits,
            "granularity": "per-channel" if spec0.group_size == 0 else f"g{spec0.group_size}",
            "phi": phi_label(spec0.phi_format, spec0.bits),
            "activations": ("int8 per-token" if spec0.act_per_token else "int8 per-tensor") if spec0.act_bits == 8
            else "bf16",
            "merge": wl.merge, "parallelism": "replicas" if world > 1 else "single",
            "launch": "eager library calls" if args.no_graph else "CUDA graph replay of each step's library calls",
            "l2": f"inputs rotate over {args.sets} device copies ({in_bytes / 2**20:.0f} MiB) > L2"}


# --------------------------------------------------------------------------- GPU arm
class GpuWorkload:
    """Device-resident layers of a workload, prepared through the library (range
    setting and downcast), with `sets` distinct copies of the step inputs."""

    def __init__(self, wl, sets: int, seed: int = 0):
        import numpy as np
        import torch
        from paper_2406_06385_gb300 import lrqat as LQ
        from paper_2406_06385_gb300 import workloads as WL
        self.wl = wl
        self.T = wl.tokens
        self.layers = []
        dev = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a)).cuda()
        for li, spec in enumerate(wl.layers):
            d = WL.make_layer(spec, self.T, seed=seed, layer_index=li)
            W0 = dev(d.W0)
            ng = spec.k // spec.group_size if spec.group_size else 1
            s = torch.empty((spec.m, ng) if spec.group_size else (spec.m,), dtype=torch.float32, device="cuda")
            z = torch.empty_like(s) if spec.asym else None   # zero offsets (asymmetric weights)
            L = LQ.Layer.from_spec(spec, z.data_ptr() if spec.asym else 0)
            LQ.range_minmax(L, W0, s)
            if spec.phi_format == WL.PHI_INT_PACKED:
                phi0 = torch.empty((spec.m, spec.k // 2), dtype=torch.uint8, device="cuda")
            elif spec.phi_format in (WL.PHI_BF16, WL.PHI_FP16):
                phi0 = torch.empty((spec.m, spec.k), dtype=torch.int16, device="cuda")
            else:
                phi0 = torch.empty((spec.m, spec.k), dtype=torch.int8, device="cuda")
            LQ.downcast(L, W0, s, phi0)
            del W0
            X = [dev(d.X_bits) for _ in range(sets)]
            dY = [dev(d.dY_bits) for _ in range(sets)]
            s_x = None
            if spec.act_bits == 8 and not spec.act_per_token:
                sx = np.float32(np.float32(np.abs(d.X).max()) / np.float32(127.0))
                s_x = torch.tensor([sx], dtype=torch.float32, device="cuda")
            lay = dict(spec=spec, L=L, z=z, phi0=phi0, s=s, A=dev(d.A_bits), B=dev(d.B_bits), X=X, dY=dY, s_x=s_x,
                       X_host=d.X_bits, dY_host=d.dY_bits,
                       Y=torch.empty((self.T, spec.m), dtype=torch.int16, device="cuda"),
                       dX=torch.empty((self.T, spec.k), dtype=torch.int16, device="cuda"),
                       dA=torch.empty((spec.m, spec.r), dtype=torch.float32, device="cuda"),
                       dB=torch.empty((spec.r, spec.k), dtype=torch.float32, device="cuda"),
                       ds=torch.empty_like(s))
            if spec.act_bits == 8:
                # the step quantizes X once and runs the forward and the backward on its codes
                lay["Xq"] = torch.empty((self.T, spec.k), dtype=torch.int16, device="cuda")
                lay["xmask"] = None if spec.act_per_token else torch.empty(
                    (spec.k, (self.T + 31) // 32), dtype=torch.int32, device="cuda")
            lay["wsf"] = torch.empty(max(LQ.fwd_workspace_bytes(L, self.T), 16), dtype=torch.uint8, device="cuda")
            lay["wsb"] = torch.empty(LQ.bwd_workspace_bytes(L, self.T), dtype=torch.uint8, device="cuda")
            self.layers.append(lay)
            if wl.merge:
                lay["WZ"] = torch.empty((spec.m, spec.k), dtype=torch.int8, device="cuda")
        torch.cuda.synchronize()
        self.sets = sets

    def step(self, i: int, X=None, dY=None, outs=None):
        """One fwd+bwd pass over every layer; X, dY, outs: optional per-layer overrides (keyed by id(layer))."""
        from paper_2406_06385_gb300 import lrqat as LQ
        j = i % self.sets
        for lay in self.layers:
            x = lay["X"][j] if X is None else X[id(lay)]
            dy = lay["dY"][j] if dY is None else dY[id(lay)]
            o = lay if outs is None else outs[id(lay)]
            if "Xq" in lay:
                # int8 activations: one quantizer pass per step feeds both GEMM passes
                LQ.act_quant(lay["L"], self.T, x, lay["s_x"], lay["Xq"], lay["xmask"])
                LQ.linear_fwd_quantized(lay["L"], self.T, lay["Xq"], lay["phi0"], lay["s"], lay["A"], lay["B"],
                                        lay["s_x"], o["Y"], lay["wsf"])
                LQ.linear_bwd_quantized(lay["L"], self.T, dy, lay["Xq"], lay["xmask"], lay["phi0"], lay["s"],
                                        lay["A"], lay["B"], lay["s_x"], o["dX"], o["dA"], o["dB"], o["ds"], False,
                                        lay["wsb"])
            else:
                LQ.linear_fwd(lay["L"], self.T, x, lay["phi0"], lay["s"], lay["A"], lay["B"], lay["s_x"], o["Y"],
                              lay["wsf"])
                LQ.linear_bwd(lay["L"], self.T, dy, x, lay["phi0"], lay["s"], lay["A"], lay["B"], lay["s_x"],
                              o["dX"], o["dA"], o["dB"], o["ds"], False, lay["wsb"])
            if self.wl.merge:
                LQ.merge(lay["L"], lay["phi0"], lay["A"], lay["B"], lay["WZ"])


def capture_steps(gw):
    """One CUDA graph of gw.step(j) per input set j, captured after an eager pass over
    every set (first calls configure kernels and cache device data).  Replaying them
    runs the same library kernels without the per-call host work and launch gaps."""
    import torch
    for j in range(gw.sets):
        gw.step(j)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graphs = []
    with torch.cuda.stream(side):
        for j in range(gw.sets):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                gw.step(j)
            graphs.append(g)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    return lambda i: graphs[i % gw.sets].replay()


def time_steps(fn, steps: int, warmup: int):
    import torch
    for i in range(warmup):
        fn(i)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for i in range(steps):
        fn(i)
    e1.record()
    e1.synchronize()
    torch.cuda.synchronize()
    barrier()
    return e0.elapsed_time(e1)


def run_gpu(args):
    import torch
    from paper_2406_06385_gb300 import lrqat as LQ
    from paper_2406_06385_gb300 import workloads as WL
    from paper_2406_06385_gb300.build import build

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    if rank == 0:
        build()
    barrier()
    LQ.lib()
    wl = WL.workload(args.workload)
    T = wl.tokens
    flops = wl.flops_fwd_bwd()
    gw = GpuWorkload(wl, sets=args.sets)
    props = torch.cuda.get_device_properties(torch.cuda.current_device())
    uuid = getattr(props, "uuid", None)
    uuid = f"GPU-{uuid}" if uuid is not None and not str(uuid).startswith("GPU-") else (str(uuid) if uuid else None)

    # 1) device-resident timed region (the headline value): each step's library calls,
    #    replayed from CUDA graphs (eager calls with --no-graph)
    step_fn = gw.step if args.no_graph else capture_steps(gw)
    with ClockSampler(uuid) as clocks:
        ms = time_steps(step_fn, args.steps, args.warmup)
    LQ.get_device_status()
    ms, units = aggregate_over_ranks(ms, float(T * args.steps))
    value = units / (ms / 1e3)
    ms_per_step = ms / args.steps

    # 2) traced pass: per-kernel device time on the launching stream, launch counts
    LQ.trace_enable(True)
    ms_traced = time_steps(gw.step, args.steps, 0)
    trace = LQ.trace_read()
    LQ.trace_enable(False)
    LQ.get_device_status()
    launches = sum(n for n, _ in trace.values())
    dom = max((k for k in trace if k in GEMM_KERNELS), key=lambda k: trace[k][1])
    n_dom, ms_dom = trace[dom]
    # algorithmic work of the kernel: 2 T m k per launch (one launch per layer per step)
    dom_flops_total = (n_dom / len(gw.layers)) * sum(2.0 * T * l["spec"].m * l["spec"].k for l in gw.layers)
    dom_flops = dom_flops_total / n_dom
    avg_ms = ms_dom / n_dom
    dom_bytes = sum(kernel_bytes(T, l["spec"]) for l in gw.layers) / len(gw.layers)
    peaks, peak_src = load_peaks()
    achieved = dom_flops_total / (ms_dom / 1e3) / 1e12
    traffic = profiled_traffic(dom, args.workload)

    # 3) end to end: pinned host inputs in, the step's result out, inside the timed region.  The inputs
    #    are every layer's X and dY; the result is what the step produces for the optimizer, the
    #    gradients dA, dB, ds of every layer (Y and dX stay on the device, where a network's adjacent
    #    layers consume them).  Like a training loop's data prefetch, step i+1's inputs are copied on a
    #    second stream while step i computes, and step i's gradients are read back on a third stream
    #    while step i+1 computes (device inputs and outputs double-buffered); every step's copies are
    #    inside the timed region.
    import numpy as np
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a.view(np.int16))).pin_memory()
    hx = {id(l): pin(l["X_host"]) for l in gw.layers}
    hdy = {id(l): pin(l["dY_host"]) for l in gw.layers}
    out_names = ("Y", "dX", "dA", "dB", "ds")   # written by the step
    result_names = ("dA", "dB", "ds")           # read back to the host
    d_in = [({id(l): l["X"][0] for l in gw.layers}, {id(l): l["dY"][0] for l in gw.layers}),
            ({id(l): torch.empty_like(l["X"][0]) for l in gw.layers},
             {id(l): torch.empty_like(l["dY"][0]) for l in gw.layers})]
    d_out = [{id(l): {n: l[n] for n in out_names} for l in gw.layers},
             {id(l): {n: torch.empty_like(l[n]) for n in out_names} for l in gw.layers}]
    h_out = [{id(l): {n: torch.empty(l[n].shape, dtype=l[n].dtype, pin_memory=True) for n in result_names}
              for l in gw.layers} for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in list(hx.values()) + list(hdy.values()))
    d2h = sum(t.numel() * t.element_size() for l in gw.layers for t in h_out[0][id(l)].values())
    comp = torch.cuda.current_stream()
    # X and dY go up on two streams (two copy engines), the result comes back on a third
    s_in, s_in2, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_comp = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def copy_in(b):
        s_in2.wait_stream(s_in)
        with torch.cuda.stream(s_in2):
            for l in gw.layers:
                d_in[b][1][id(l)].copy_(hdy[id(l)], non_blocking=True)
        with torch.cuda.stream(s_in):
            for l in gw.layers:
                d_in[b][0][id(l)].copy_(hx[id(l)], non_blocking=True)
            s_in.wait_stream(s_in2)
            ev_in[b].record(s_in)

    def e2e_run(steps: int):
        s_in.wait_stream(comp)
        s_out.wait_stream(comp)
        copy_in(0)
        for i in range(steps):
            b = i % 2
            if i + 1 < steps:
                if i >= 1:
                    s_in.wait_event(ev_comp[1 - b])     # buffers 1-b were last read by step i-1
                copy_in(1 - b)
            comp.wait_event(ev_in[b])
            if i >= 2:
                comp.wait_event(ev_out[b])               # outputs b of step i-2 have been read back
            gw.step(0, X=d_in[b][0], dY=d_in[b][1], outs=d_out[b])
            ev_comp[b].record(comp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_comp[b])
                for l in gw.layers:
                    for n in result_names:
                        h_out[b][id(l)][n].copy_(d_out[b][id(l)][n], non_blocking=True)
                ev_out[b].record(s_out)
        comp.wait_stream(s_out)

    def time_e2e(steps: int, warmup: int) -> float:
        e2e_run(warmup)
        torch.cuda.synchronize()
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(comp)
        e2e_run(steps)
        e1.record(comp)
        e1.synchronize()
        torch.cuda.synchronize()
        barrier()
        return e0.elapsed_time(e1)

    e2e_steps = max(3, min(args.steps, int(3000.0 / max(ms_per_step, 1e-3) / 2)))
    ms_e2e = time_e2e(e2e_steps, 2)
    ms_e2e, units_e2e = aggregate_over_ranks(ms_e2e, float(T * e2e_steps))

    clk = clocks.summary()
    if rank != 0:
        return None
    # The burst peak (a GEMM timed alone at full clock) is the denominator unless the clock
    # record of the timed region shows the power cap or clocks below the maximum; then the
    # sustained peak (a seconds-long GEMM loop under the power cap) is.
    kind = peak_kind(clk)
    peak = peaks["bf16_tflops" if kind == "burst" else "bf16_tflops_sustained"]
    cfg = workload_config(wl, args, world)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded normal weights/activations, LLaMA-shaped layers)",
        "config": cfg,
        "tflops": flops * args.steps * world / (ms / 1e3) / 1e12,
        "frac_of_bf16_peak": {"value": flops * args.steps * world / (ms / 1e3) / 1e12 / peak, "peak_kind": kind,
                              "burst": flops * args.steps * world / (ms / 1e3) / 1e12 / peaks["bf16_tflops"],
                              "sustained": flops * args.steps * world / (ms / 1e3) / 1e12 / peaks["bf16_tflops_sustained"],
                              "peaks": peak_src},
        "roofline": {"kernel": dom, "bound": "tensor", "achieved": achieved, "peak": peak,
                     "unit": "TFLOP/s", "frac": achieved / peak, "traffic": traffic,
                     "peak_kind": f"bf16 dense, {kind} ({peak_src})",
                     "frac_sustained": achieved / peaks["bf16_tflops_sustained"],
                     "launch_ms": avg_ms, "flops_per_launch": dom_flops,
                     "algorithmic_bytes_per_launch": dom_bytes},
        "kernels": {k: {"launches": n, "total_ms": t, "share": t / sum(v[1] for v in trace.values())}
                    for k, (n, t) in sorted(trace.items(), key=lambda kv: -kv[1][1])},
        "traced_ms_per_step": ms_traced / args.steps,
        "gpu_launches": launches,
        "e2e": {"value": units_e2e / (ms_e2e / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps, "h2d": "X and dY of every layer",
                "d2h": "dA, dB and ds of every layer (the step's result)"},
        "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"],
                   "samples": clk["samples"], "power_w_max": clk.get("power_w_max")},
    }
    if world == 1 and not args.no_cpu_baseline:
        # the oracle leg: the timed CPU baseline, then the GPU outputs of the first layer
        # checked against the oracle on samples (not part of any timed region)
        line["cpu_baseline"] = cpu_baseline(wl, budget_s=args.cpu_budget)
        line["cpu_baseline"]["single_thread"] = cpu_baseline_single_thread(args.workload, args.cpu_budget / 3)
        try:
            line["parity"] = sampled_parity(gw)
        except Exception as e:   # reported in the line; the timed numbers above stand
            line["parity"] = {"ok": False, "error": f"{type(e).__name__}: {e}"}
    return line


# --------------------------------------------------------------------------- CPU oracle
def _oracle_sample(wl, rows: int, tokens: int):
    """One layer's data cut to `rows` output channels and `tokens` tokens (a smaller
    LR-QAT layer with the same per-element arithmetic), prepared for the oracle."""
    import numpy as np
    import oracle as O
    from paper_2406_06385_gb300 import workloads as WL
    spec = wl.layers[0]
    d = WL.make_layer(spec, wl.tokens, seed=0, layer_index=0)
    OL = O.Layer(spec.m, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format, spec.act_bits,
                 spec.act_per_token)
    if spec.asym:   # asymmetric weights: zero offsets from asymmetric range setting
        s0, z0 = O.minmax_range_asym(d.W0, OL)
        phi0 = O.downcast(d.W0, s0, OL, z0)
        z0 = z0[:rows]
    else:
        s0, z0 = O.minmax_scale(d.W0, OL), None
        phi0 = O.downcast(d.W0, s0, OL)
    sub = O.Layer(rows, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format, spec.act_bits,
                  spec.act_per_token)
    X = d.X[:tokens]
    s_x = (float(np.float32(np.abs(d.X).max()) / np.float32(127.0))
           if spec.act_bits == 8 and not spec.act_per_token else None)
    return dict(OL=sub, phi0=phi0[:rows], s=s0[:rows], z=z0, A=d.A[:rows], B=d.B, X=X, dY=d.dY[:tokens, :rows],
                s_x=s_x, frac=rows / spec.m, tokens=tokens, m=spec.m)


def _oracle_step(smp):
    import oracle as O
    O.linear_fwd(smp["X"], smp["phi0"], smp["s"], smp["A"], smp["B"], smp["OL"], smp["s_x"], smp["z"])
    O.linear_bwd(smp["dY"], smp["X"], smp["phi0"], smp["s"], smp["A"], smp["B"], smp["OL"], smp["s_x"], smp["z"])


def _calibrated_sample(wl, budget_s: float):
    """A (rows, tokens) cut of the workload's first layer whose oracle step takes
    between budget_s / 2 and budget_s seconds (cost roughly doubles with either)."""
    rows, tokens = 128, min(256, wl.tokens)
    smp = _oracle_sample(wl, rows, tokens)
    t0 = time.perf_counter()
    _oracle_step(smp)
    t = time.perf_counter() - t0
    m = wl.layers[0].m
    while t < budget_s / 2:
        if tokens < wl.tokens:
            tokens = min(wl.tokens, tokens * 2)
        elif rows < m:
            rows = min(m, rows * 2)
        else:
            break
        t *= 2
    return _oracle_sample(wl, rows, tokens)


def cpu_baseline(wl, budget_s: float = 15.0):
    """The oracle as it stands, on this host's cores, over a bounded sample of the workload."""
    smp = _calibrated_sample(wl, budget_s / 3)
    reps = 0
    t0 = time.perf_counter()
    while True:
        _oracle_step(smp)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= budget_s or reps >= 20:
            break
    nlayers = len(wl.layers)
    value = smp["tokens"] * smp["frac"] * reps / dt / nlayers
    return {"value": value, "unit": UNIT, "cores": len(os.sched_getaffinity(0)), "kind": "oracle",
            "seconds": dt,
            "sample": (f"{reps} oracle fwd+bwd steps of the first layer ({wl.layers[0].m}x{wl.layers[0].k}) cut to "
                       f"{smp['OL'].m} output channels and {smp['tokens']} tokens (float64 numpy, BLAS on all host "
                       f"cores); value = tokens x (rows/m) x steps / time / {nlayers} layer(s), i.e. full-workload "
                       f"tokens/s assuming equal per-layer cost")}


def cpu_baseline_single_thread(workload: str, budget_s: float = 5.0):
    """The oracle with its BLAS and OpenMP pools pinned to one thread and the process to one
    core, over its own bounded sample (a child process: the thread counts must be set before
    numpy loads)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               BLIS_NUM_THREADS="1", VECLIB_MAXIMUM_THREADS="1", NUMEXPR_NUM_THREADS="1")
    code = (f"import sys, json; sys.path.insert(0, {ROOT!r}); import bench; "
            f"print(json.dumps(bench._single_thread_child({workload!r}, {float(budget_s)!r})))")
    try:
        r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                           timeout=max(120.0, 20 * budget_s))
        return json.loads(r.stdout.strip().splitlines()[-1])
    except (subprocess.TimeoutExpired, ValueError, IndexError) as e:
        return {"unavailable": f"single-thread oracle run failed: {type(e).__name__}"}


def _single_thread_child(workload: str, budget_s: float):
    try:
        os.sched_setaffinity(0, {sorted(os.sched_getaffinity(0))[0]})
    except (AttributeError, OSError):
        pass
    from paper_2406_06385_gb300 import workloads as WL
    wl = WL.workload(workload)
    smp = _calibrated_sample(wl, budget_s / 2)
    reps = 0
    t0 = time.perf_counter()
    while True:
        _oracle_step(smp)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= budget_s or reps >= 10:
            break
    nlayers = len(wl.layers)
    return {"value": smp["tokens"] * smp["frac"] * reps / dt / nlayers, "unit": UNIT, "cores": 1, "kind": "oracle",
            "seconds": dt,
            "sample": (f"{reps} oracle fwd+bwd steps of the first layer cut to {smp['OL'].m} output channels and "
                       f"{smp['tokens']} tokens, BLAS and OpenMP pinned to one thread on one core")}


def sampled_parity(gw, n_tokens: int = 24, n_rows: int = 6, n_cols: int = 6):
    """The first layer's outputs of the timed step against the oracle, the way the full-size
    parity tests check them: every integer code of W_hat (bit for bit outside near-ties,
    read through a forward with X = I and s = 1, which turns Y into the codes), Y and dX at
    sampled token rows, dA and ds at sampled weight rows, dB at sampled weight columns
    (relative Frobenius errors; tolerances 1e-2 for Y, dX and 2e-2 for the gradients)."""
    import numpy as np
    import torch
    import oracle as O
    from paper_2406_06385_gb300 import lrqat as LQ
    from paper_2406_06385_gb300 import workloads as WL
    lay = gw.layers[0]
    spec, T, L = lay["spec"], gw.T, lay["L"]
    f32 = lambda t: WL.bf16_to_f32(t.cpu().numpy().view(np.uint16))
    # outputs of the last timed step (every input set holds the same data)
    Y, dX = lay["Y"], lay["dX"]
    dA, dB, ds = lay["dA"].cpu().numpy(), lay["dB"].cpu().numpy(), lay["ds"].cpu().numpy()
    # the codes: X = I_k, s = 1, no activation quantizer
    Lc = LQ.Layer.from_spec(spec, lay["z"].data_ptr() if lay["z"] is not None else 0)
    Lc.act_bits, Lc.act_per_token = 0, 0
    eye = torch.eye(spec.k, dtype=torch.bfloat16, device="cuda").view(torch.int16)
    yc = torch.empty((spec.k, spec.m), dtype=torch.int16, device="cuda")
    wsc = torch.empty(max(LQ.fwd_workspace_bytes(Lc, spec.k), 16), dtype=torch.uint8, device="cuda")
    LQ.linear_fwd(Lc, spec.k, eye, lay["phi0"], torch.ones_like(lay["s"]), lay["A"], lay["B"], None, yc, wsc)
    LQ.get_device_status()
    codes_gpu = f32(yc).T
    del eye, yc, wsc

    d = WL.make_layer(spec, T, seed=0, layer_index=0)
    OL = O.Layer(spec.m, spec.k, spec.r, spec.alpha, spec.bits, spec.group_size, spec.phi_format, spec.act_bits,
                 spec.act_per_token, spec.u_bf16)
    if spec.asym:
        s0, z0 = O.minmax_range_asym(d.W0, OL)
        phi0 = O.downcast(d.W0, s0, OL, z0)
    else:
        s0, z0 = O.minmax_scale(d.W0, OL), None
        phi0 = O.downcast(d.W0, s0, OL)
    fq = O.fake_quant_weight(phi0, s0, d.A, d.B, OL, z0)
    exempt = O.near_tie(fq["u"])
    mism = int(((codes_gpu != fq["cz"]) & ~exempt).sum())
    s_x = None
    if spec.act_bits == 8 and spec.act_per_token:
        _, Xh, Mx, _ = O.act_quant_per_token(d.X)
    elif spec.act_bits == 8:
        s_x = float(np.float32(np.abs(d.X).max()) / np.float32(127.0))
        _, Xh, Mx = O.act_quant(d.X, s_x)
    else:
        Xh, Mx = d.X.astype(np.float64), None
    dYf = d.dY.astype(np.float64)
    lr = OL.alpha / OL.r
    ts = WL.token_sample(T, n_tokens, seed=1)
    tsel = torch.as_tensor(ts, device="cuda")
    dX_ref = dYf[ts] @ fq["W_hat"]
    if Mx is not None:
        dX_ref = dX_ref * Mx[ts]
    errs = {"Y": O.rel_fro(f32(Y[tsel]), Xh[ts] @ fq["W_hat"].T), "dX": O.rel_fro(f32(dX[tsel]), dX_ref)}
    rows = WL.token_sample(spec.m, n_rows, seed=2)
    G_rows = dYf[:, rows].T @ Xh
    s_full = O.expand_scale(s0, OL)
    errs["dA"] = O.rel_fro(dA[rows], lr * ((G_rows * s_full[rows] * fq["M"][rows]) @ d.B.astype(np.float64).T))
    Gc = G_rows * fq["cz"][rows]
    ds_ref = Gc.sum(axis=1) if spec.group_size == 0 else Gc.reshape(len(rows), -1, spec.group_size).sum(axis=2)
    errs["ds"] = O.rel_fro(ds.reshape((spec.m, -1) if spec.group_size else (spec.m,))[rows], ds_ref)
    cols = WL.token_sample(spec.k, n_cols, seed=3)
    G_cols = dYf.T @ Xh[:, cols]
    errs["dB"] = O.rel_fro(dB[:, cols], lr * (d.A.astype(np.float64).T @ (G_cols * s_full[:, cols] * fq["M"][:, cols])))
    tol = {"Y": 1e-2, "dX": 1e-2, "dA": 2e-2, "dB": 2e-2, "ds": 2e-2}
    return {"layer": f"{spec.name}:{spec.m}x{spec.k}", "codes_checked": int(fq["cz"].size), "code_mismatches": mism,
            "near_tie_exempt": int(exempt.sum()), "rel_err": errs,
            "ok": mism == 0 and all(errs[k] <= tol[k] for k in tol),
            "sample": f"{len(ts)} token rows (Y, dX), {len(rows)} weight rows (dA, ds), {len(cols)} weight columns (dB)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return None
    from paper_2406_06385_gb300 import workloads as WL
    wl = WL.workload(args.workload)
    per_step = max(0.02, min(10.0, 150.0 / max(1, args.steps + args.warmup)))
    smp = _calibrated_sample(wl, per_step)
    for _ in range(args.warmup):
        _oracle_step(smp)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _oracle_step(smp)
    dt = time.perf_counter() - t0
    nlayers = len(wl.layers)
    value = smp["tokens"] * smp["frac"] * args.steps / dt / nlayers
    cores = len(os.sched_getaffinity(0))
    sample = (f"each step: first layer ({wl.layers[0].m}x{wl.layers[0].k}) cut to {smp['OL'].m} output channels "
              f"and {smp['tokens']} tokens; value = tokens x (rows/m) / time / {nlayers} layer(s)")
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(wl, args, world), "impl": "reference",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main(argv=None):
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=("lrqat", "reference"), default="lrqat")
    p.add_argument("--workload", default="llama2_13b_layer",
                   help="default: all seven projections of a LLaMA-2-13B decoder layer, T = 16384, with merge")
    p.add_argument("--sets", type=int, default=4, help="distinct device copies of the step inputs (L2 rotation)")
    p.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-graph", action="store_true", help="time eager library calls instead of CUDA graph replays")
    args = p.parse_args(argv)
    if args.warmup < 3:
        p.error("--warmup must be >= 3")
    line = run_reference(args) if args.impl == "reference" else run_gpu(args)
    if line is not None:
        print(json.dumps(line), flush=True)
    try:
        import torch.distributed as dist
        if dist.is_available() and dist.is_initialized():
            dist.destroy_process_group()
    except Exception:
        pass


if __name__ == "__main__":
    main()
