"""Host-side logic of bench.py: multi-rank aggregation over gloo (world size 2),
clock-sample parsing, the CPU reference arm's JSON line, and the traffic lookup."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _agg_worker(rank, world, port, q):
    import torch.distributed as dist
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        q.put((rank, bench.aggregate_over_ranks(10.0 + rank, 100.0 * (rank + 1))))
        bench.barrier()
    finally:
        dist.destroy_process_group()


def test_aggregate_over_ranks_gloo_world2():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_agg_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = dict(q.get(timeout=10) for _ in range(2))
    # slowest rank's time, summed units, identical on both ranks
    assert res[0] == res[1] == (11.0, 300.0)


def test_aggregate_without_process_group_is_identity():
    assert bench.aggregate_over_ranks(3.5, 7.0) == (3.5, 7.0)


def test_clock_summary_parsing(tmp_path):
    cs = bench.ClockSampler("GPU-abc")
    cs.path = str(tmp_path / "c.csv")
    with open(cs.path, "w") as f:
        f.write("0, GPU-abc, 1800, 2070, 900.5, 99, 0x0, Not Active, Not Active, Not Active, Active\n")
        f.write("0, GPU-abc, 1900, 2070, 1000.0, 100, 0x0, Not Active, Not Active, Not Active, Not Active\n")
        f.write("0, GPU-abc, 600, 2070, 100.0, 0, 0x0, Not Active, Not Active, Not Active, Not Active\n")
        f.write("1, GPU-zzz, 100, 2070, 10.0, 100, 0x0, Active, Active, Active, Active\n")
    s = cs.summary()
    assert s["sm_mhz"] == 1850 and s["sm_max_mhz"] == 2070 and s["samples"] == 2
    assert s["reasons"] == ["sw_power_cap"]


def test_traffic_lookup_requires_matching_source(tmp_path, monkeypatch):
    prof = tmp_path / "profiles"
    prof.mkdir()
    h = bench.kernel_source_hash("fused_dw")
    (prof / "fused_dw_w.md").write_text(f"dram_bytes_per_launch: 1.5e8\nsource_sha256_16: {h}\n")
    (prof / "fused_fwd_w.md").write_text("dram_bytes_per_launch: 2e8\nsource_sha256_16: 0000000000000000\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    csrc = os.path.join(tmp_path, "paper_2406_06385_gb300", "csrc")
    os.makedirs(csrc)
    for name in os.listdir(os.path.join(ROOT, "paper_2406_06385_gb300", "csrc")):
        with open(os.path.join(ROOT, "paper_2406_06385_gb300", "csrc", name), "rb") as src:
            open(os.path.join(csrc, name), "wb").write(src.read())
    assert bench.profiled_traffic("fused_dw", "w") == 1.5e8
    assert bench.profiled_traffic("fused_fwd", "w") is None
    assert bench.profiled_traffic("fused_dx", "w") is None


def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "3"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["metric"] == bench.METRIC


def test_reference_arm_names_the_gpu_arms_config():
    """Both arms print the same `config` object for the same arguments (workload, shapes,
    quantizer settings, launch mode and input rotation), so their lines describe one workload."""
    import argparse
    from paper_2406_06385_gb300 import workloads as WL
    args = argparse.Namespace(sets=4, no_graph=False)
    wl = WL.workload("llama2_13b_layer")
    cfg = bench.workload_config(wl, args, 1)
    assert cfg["workload"] == "llama2_13b_layer" and cfg["tokens"] == 16384 and len(cfg["layers"]) == 7
    assert cfg["merge"] is True and cfg["phi"] == "Q4.4 int8" and cfg["granularity"] == "per-channel"
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "3"], capture_output=True, text=True, timeout=600)
    d = json.loads(r.stdout.strip().splitlines()[-1])
    assert d["config"] == bench.workload_config(WL.workload("tiny"), args, 1)


def test_warmup_below_three_is_rejected():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--warmup", "2"],
                       capture_output=True, text=True, timeout=120, cwd=ROOT)
    assert r.returncode != 0


def test_peak_kind_follows_the_clock_record():
    """Burst peak at full clock without the power cap; sustained otherwise."""
    assert bench.peak_kind({"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}) == "burst"
    assert bench.peak_kind({"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}) == "sustained"
    assert bench.peak_kind({"sm_mhz": 1462.0, "sm_max_mhz": 2070.0, "reasons": []}) == "sustained"
    assert bench.peak_kind({"sm_mhz": None, "sm_max_mhz": None, "reasons": []}) == "burst"


def test_algorithmic_bytes_of_a_gemm_launch():
    """Two bf16 token operands of T rows, the stored base once (int8 here) and the adapters."""
    from paper_2406_06385_gb300 import workloads as WL
    spec = WL.workload("llama2_7b_attn").layers[0]
    T = 8192
    assert bench.kernel_bytes(T, spec) == 2 * T * 8192 + 4096 * 4096 + 2 * 32 * 8192


def test_single_thread_baseline_child_runs_on_one_core():
    d = bench.cpu_baseline_single_thread("tiny", budget_s=0.5)
    assert d["cores"] == 1 and d["value"] > 0 and d["kind"] == "oracle", d
