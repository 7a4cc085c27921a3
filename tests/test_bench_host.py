"""bench.py host logic: the workload's FLOP counts and the replica aggregation under gloo."""
import os
import socket
import subprocess
import sys


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def test_workload_flops_match_config():
    wl = bench.workload("1.3b")
    # 4 Nq Nk d H: full over 18 frames + chunk, local over 6 frames + chunk
    assert wl["nq"] == 4680 and wl["nk_full"] == 32760 and wl["nk_local"] == 14040
    assert abs(wl["flops_full"] / 1e12 - 0.942) < 5e-4
    assert abs(wl["flops_local"] / 1e12 - 0.404) < 5e-4
    assert wl["flops_dual"] == wl["flops_full"]
    wl14 = bench.workload("14b")
    assert wl14["D"] == 5120 and abs(wl14["flops_local"] / 1e12 - 1.346) < 1e-3


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


WORKER = r"""
import os, sys, torch, torch.distributed as dist
dist.init_process_group("gloo")
r, w = dist.get_rank(), dist.get_world_size()
# each replica reports its own time; the job's time is the max, value sums the replicas
t = torch.tensor([10.0 + r])
dist.all_reduce(t, op=dist.ReduceOp.MAX)
assert t.item() == 10.0 + (w - 1)
dist.barrier()
if r == 0:
    print("ok", w, t.item())
dist.destroy_process_group()
"""


def test_replica_max_over_ranks_gloo(tmp_path):
    f = tmp_path / "w.py"
    f.write_text(WORKER)
    env = dict(os.environ, MASTER_ADDR="127.0.0.1", MASTER_PORT=str(_free_port()))
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={env['MASTER_PORT']}", str(f)]
    r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr[-2000:]
    assert "ok 2 11.0" in r.stdout


def test_reference_arm_skips_non_zero_ranks(capsys):
    class A:
        model = "1.3b"
        ref_rows = 2
        steps = 1
        warmup = 0
    bench.run_reference(A, rank=1, world=2)
    assert capsys.readouterr().out == ""


def test_clock_rejection_rule():
    import bench
    ok = dict(sm_mhz=2070.0, sm_max_mhz=2070.0, reasons=[], samples=5)
    assert not bench.clock_rejected(ok) and not bench.clock_rejected(None)
    assert not bench.clock_rejected(dict(ok, reasons=["sw_power_cap"], sm_mhz=1900.0))
    assert bench.clock_rejected(dict(ok, reasons=["hw_slowdown"]))
    assert bench.clock_rejected(dict(ok, reasons=["sw_thermal_slowdown", "sw_power_cap"]))
    assert bench.clock_rejected(dict(ok, sm_mhz=1400.0))              # stuck low, no reason
    assert not bench.clock_rejected(dict(ok, sm_mhz=1400.0, reasons=["sw_power_cap"]))


def test_roofline_traffic_only_for_the_captured_source_and_shape(monkeypatch):
    import bench
    pk = dict(bf16=2000.0, bf16_sustained=1600.0, source="measured")
    r = bench.roofline_entry("1.3b", 1500.0, pk)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["frac"] == 0.75 and r["frac_of_sustained"] == round(1500 / 1600, 4)
    captured = bench.ATTN_TRAFFIC["source_sha256_16"] == bench.attn_source_sha()
    assert r["traffic"] == (bench.ATTN_TRAFFIC["bytes"] if captured else None)
    # another model shape, or a changed kernel source: no traffic figure
    assert bench.roofline_entry("14b", 1500.0, pk)["traffic"] is None
    monkeypatch.setattr(bench, "attn_source_sha", lambda: "0" * 16)
    assert bench.roofline_entry("1.3b", 1500.0, pk)["traffic"] is None


def test_ls_flops_method_and_tile_work():
    # method work 2T(2D^2 + D): 44.2 GFLOP for the 1.3B step (T 4680, D 1536), 490.8 for 14B
    m, t = bench.ls_flops(1536, 4680)
    assert abs(m / 1e9 - 44.18) < 0.01
    # 256 x 256 tiles: 6 x 6 grid, 21 upper tiles; scaled form one pass per tile: 21 + 36 + 21 = 78
    assert t == 78 * 2.0 * 256 * 256 * 4680
    # exact form: 21 (G) + 2 * 36 (X) + 3 * 21 (S) = 156 tile-passes
    _, te = bench.ls_flops(1536, 4680, exact=True)
    assert te == 156 * 2.0 * 256 * 256 * 4680
    m14, _ = bench.ls_flops(5120, 4680)
    assert abs(m14 / 1e9 - 490.8) < 0.1
    # a width with no 256 tiling falls back to 128 x 128 tiles
    _, t384 = bench.ls_flops(384, 10, exact=True)
    assert t384 == (6 + 2 * 9 + 3 * 6) * 2.0 * 128 * 128 * 10
    _, t384s = bench.ls_flops(384, 10)
    assert t384s == (6 + 9 + 6) * 2.0 * 128 * 128 * 10


def test_modes_rates_and_fractions():
    import numpy as np
    wl = bench.workload("1.3b")
    pk = dict(bf16=2000.0, bf16_sustained=1600.0, hbm=7000.0, source="measured")
    seg = np.array([[0.6, 0.3, 0.62, 0.08, 0.03]] * 4)
    m = bench.modes_of(seg, wl, pk)
    assert abs(m["full"]["tflops"] - wl["flops_full"] / 0.6e-3 / 1e12) < 1e-3
    assert abs(m["full"]["frac"] - m["full"]["tflops"] / 2000.0) < 1e-4
    assert abs(m["ls_accumulate"]["method_tflops"] - 44.18e9 / 0.08e-3 / 1e12) < 0.5
    gbs = 3 * 2 * 2 * 4680 * 1536 * 2 / 0.03e-3 / 1e9
    assert abs(m["kv_append"]["gbs"] - gbs) < 0.01 and abs(m["kv_append"]["frac"] - gbs / 7000.0) < 1e-4


def test_nvml_sampler_window_and_reasons():
    # the summary keeps only samples inside the timed window and maps the reason bits
    s = bench.NvmlSampler.__new__(bench.NvmlSampler)
    s.t, s.run, s.period = None, False, 0.004
    s.samples = [(0.5, 1200, 2070, 100000, 0x1),           # before the region: idle
                 (1.0, 2070, 2070, 900000, 0x0), (1.01, 2040, 2070, 950000, 0x4),
                 (1.02, 2070, 2070, 990000, 0x0), (2.0, 1100, 2070, 100000, 0x8)]   # after it
    c = s.stop(1.0, 1.5)
    assert c["samples"] == 3 and c["sm_mhz"] == 2070 and c["reasons"] == ["sw_power_cap"]
    assert c["power_w_max"] == 990.0
    assert s.stop(5.0, 6.0) is None
