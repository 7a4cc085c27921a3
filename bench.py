"""Chunk-step benchmark of the ISPA hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--model 1.3b|14b]

One step = one pass of the whole hot path over one chunk of a 1.3B-shaped
layer stack (12 heads x 128, 1560 tokens/frame, 3-frame chunk = 4680 queries):
  * F-layer attention over an 18-frame ring (28080 + 4680 keys),
  * L-layer attention over its 6-frame window ring (9360 + 4680 keys),
  * warmup dual attention on an 18-frame ring (local = chunk + 6 frames, hist = 12 frames),
  * least-squares accumulation of that layer's (A_loc, A_full) over its 4680 tokens,
  * KV append of the finished chunk into all three rings (one launch).
The rings stay in steady state (each append evicts the oldest 3 frames).
value = attention FLOPs of the three modes (4*Nq*Nk*d*H each) / device time of the step.
L2 is flushed (256 MB write) between timed steps, outside the timed events.
Inputs are synthetic (seeded N(0,1) q/k/v with per-frame key offsets), bf16.

The "extras" object also times, outside the step: the two-call dual decomposition, the
solve, the W8A8 projection, the 8-bit Q K^T attention, and (unless --no-configs) the 20-step
AR rollout of the whole layer stack (30 layers at 1.3B, 40 at 14B; half F-layers over a cache
growing to 60 frames, half L-layers; batched append per step) and the warmup-to-transition
path (8 dual steps on a 24-frame cache with LS accumulation, then one solve).

Under torchrun (N > 1) every rank runs an independent replica on its own GPU
(the path has no exchange step); timing is max over ranks and value sums ranks.
--impl reference times the fp64 CPU oracle on a bounded sample of the same step.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "chunk-step attention TFLOP/s (full/local/dual) and % of GB300 dense bf16 peak"
UNIT = "TFLOP/s"

MODELS = {
    # name: (heads, head_dim, tokens/frame, chunk frames, F-ring frames, window frames)
    "1.3b": (12, 128, 1560, 3, 18, 6),
    "14b": (40, 128, 1560, 3, 18, 6),
}
MODEL_LAYERS = {"1.3b": 30, "14b": 40}   # transformer blocks of the rollout workloads (half F, half L)


def log(*a):
    print(*a, file=sys.stderr, flush=True)


# DRAM bytes of one F-layer attention launch of the 1.3B step (dram__bytes_read.sum +
# dram__bytes_write.sum from one ncu capture of that launch), valid only for the kernel source
# it was taken on: reported as null once attn.cu / ptx.cuh change.
ATTN_TRAFFIC = {"source_sha256_16": "a4d523e43ed3c924", "bytes": 242222592 + 11659008, "model": "1.3b"}


def attn_source_sha():
    import hashlib
    d = os.path.join(ROOT, "paper_2607_00712_gb300", "csrc")
    src = open(os.path.join(d, "attn.cu"), "rb").read() + open(os.path.join(d, "ptx.cuh"), "rb").read()
    return hashlib.sha256(src).hexdigest()[:16]


# GB300 datasheet dense (no 2:4 sparsity) bf16 tensor rate per GPU: 2.25 PFLOP/s.  Reported
# beside the measured cuBLAS peak so that either reading of "% of dense bf16 peak" can be taken.
NOMINAL_BF16_TFLOPS = 2250.0


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(bf16=d["bf16_tflops"], bf16_sustained=d.get("bf16_tflops_sustained"), hbm=d["hbm_gbs"],
                    source="measured")
    return dict(bf16=1900.0, bf16_sustained=1700.0, hbm=6800.0, source="fallback")


def roofline_entry(model, achieved, pk):
    """The roofline object of the F-layer attention launch: achieved TFLOP/s against the measured
    dense bf16 peak; DRAM traffic per launch only while the kernel source and the model shape are
    those the ncu counters were taken on."""
    traffic = None
    if ATTN_TRAFFIC["model"] == model and attn_source_sha() == ATTN_TRAFFIC["source_sha256_16"]:
        traffic = ATTN_TRAFFIC["bytes"]
    return dict(bound="tensor", achieved=round(achieved, 2), peak=pk["bf16"], unit="TFLOP/s",
                frac=round(achieved / pk["bf16"], 4), traffic=traffic, traffic_unit="bytes per launch",
                kernel="attn_kernel<128> (F-layer launch)", peak_source=pk["source"] + " burst bf16",
                frac_of_sustained=round(achieved / pk["bf16_sustained"], 4) if pk["bf16_sustained"] else None,
                frac_of_nominal=round(achieved / NOMINAL_BF16_TFLOPS, 4), nominal_peak=NOMINAL_BF16_TFLOPS)


def ls_flops(D, T, exact=False):
    """FLOPs of one LS accumulation: the method's own work (the upper triangles of G = A^T A and
    S = Delta^T Delta with their diagonals, and all of X = A^T Delta: 2 T (2 D^2 + D)) and the
    tile work the kernel issues (256 x 256 tiles with whole diagonal tiles, or 128 x 128 when
    D % 256 != 0; one pass per tile in the default scaled form, X in two passes and S in three
    over the bf16 hi/lo split of Delta in the exact form)."""
    method = 2.0 * T * (2.0 * D * D + D)
    tb = 256 if D % 256 == 0 else 128
    nb = D // tb
    upper = nb * (nb + 1) // 2
    passes = (1, 2, 3) if exact else (1, 1, 1)
    tile = (passes[0] * upper + passes[1] * nb * nb + passes[2] * upper) * 2.0 * tb * tb * T
    return method, tile


def attn_flops(nq, nk, d, H):
    return 4.0 * nq * nk * d * H


def workload(model):
    H, d, P, L, F, Wn = MODELS[model]
    nq = L * P
    return dict(H=H, d=d, P=P, L=L, F=F, W=Wn, nq=nq, D=H * d,
                nk_full=F * P + nq, nk_local=Wn * P + nq,
                flops_full=attn_flops(nq, F * P + nq, d, H),
                flops_local=attn_flops(nq, Wn * P + nq, d, H),
                flops_dual=attn_flops(nq, F * P + nq, d, H))


# ---------------------------------------------------------------- clocks sampler
def clock_rejected(clocks) -> bool:
    """True for a timed region that the timing rules reject: a hardware or thermal slowdown
    was active, or the SM clock sat well below its maximum with no reason reported."""
    if not clocks:
        return False
    if set(clocks["reasons"]) & {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}:
        return True
    return not clocks["reasons"] and clocks["sm_mhz"] < 0.85 * clocks["sm_max_mhz"]


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines: list[str] = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-i", str(self.idx), "-lms", "200"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def stop(self, t0: float = 0.0, t1: float = 0.0):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.t:
            self.t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return dict(sm_mhz=statistics.median(sm), sm_max_mhz=max(mx), reasons=sorted(reasons), samples=len(sm))


class NvmlSampler:
    """SM clock, power and clock-event reasons read through NVML (read-only queries) every
    `period` seconds on a thread, so that a timed region of a few tens of ms still holds several
    samples.  stop() summarises the samples taken inside [t0, t1] (host clock), the window the
    caller marks as under load.  Raises OSError if NVML cannot be loaded."""
    # nvmlClocksEventReasons bits
    BITS = {"sw_power_cap": 0x4, "hw_slowdown": 0x8, "sw_thermal_slowdown": 0x20, "hw_thermal_slowdown": 0x40}

    def __init__(self, gpu: str | int, period: float = 0.004):
        import ctypes
        self.ct = ctypes
        self.nv = ctypes.CDLL("libnvidia-ml.so.1")
        if self.nv.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        self.h = ctypes.c_void_p()
        if isinstance(gpu, str) and gpu.startswith(("GPU-", "MIG-")):
            rc = self.nv.nvmlDeviceGetHandleByUUID(gpu.encode(), ctypes.byref(self.h))
        else:
            rc = self.nv.nvmlDeviceGetHandleByIndex_v2(int(gpu), ctypes.byref(self.h))
        if rc != 0:
            raise OSError(f"no NVML handle for GPU {gpu}")
        fn = getattr(self.nv, "nvmlDeviceGetCurrentClocksEventReasons", None)
        self.reasons_fn = fn or self.nv.nvmlDeviceGetCurrentClocksThrottleReasons
        self.period = period
        self.samples: list[tuple[float, int, int, int, int]] = []
        self.run = False
        self.t = None

    def _one(self):
        ct = self.ct
        sm, mx, mw = ct.c_uint(), ct.c_uint(), ct.c_uint()
        mask = ct.c_ulonglong()
        if self.nv.nvmlDeviceGetClockInfo(self.h, 1, ct.byref(sm)) != 0:       # NVML_CLOCK_SM
            return
        self.nv.nvmlDeviceGetMaxClockInfo(self.h, 1, ct.byref(mx))
        self.nv.nvmlDeviceGetPowerUsage(self.h, ct.byref(mw))
        self.reasons_fn(self.h, ct.byref(mask))
        self.samples.append((time.perf_counter(), sm.value, mx.value, mw.value, mask.value))

    def _loop(self):
        while self.run:
            self._one()
            time.sleep(self.period)

    def start(self):
        self.run = True
        self.t = threading.Thread(target=self._loop, daemon=True)
        self.t.start()

    def stop(self, t0: float, t1: float):
        self.run = False
        if self.t:
            self.t.join(timeout=2)
        inside = [x for x in self.samples if t0 <= x[0] <= t1]
        if not inside:
            return None
        reasons = sorted(n for n, b in self.BITS.items() if any(x[4] & b for x in inside))
        return dict(sm_mhz=statistics.median(x[1] for x in inside), sm_max_mhz=max(x[2] for x in inside),
                    reasons=reasons, samples=len(inside), power_w_max=round(max(x[3] for x in inside) / 1e3, 1),
                    source=f"NVML every {self.period * 1e3:.0f} ms inside the timed region")


def make_sampler(local_rank: int):
    """NVML sampler for this rank's GPU, else the nvidia-smi one."""
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    parts = [p.strip() for p in vis.split(",") if p.strip()]
    gpu = parts[local_rank] if local_rank < len(parts) and not parts[local_rank].isdigit() else \
        physical_gpu_index(local_rank)
    try:
        return NvmlSampler(gpu)
    except (OSError, AttributeError):
        return ClockSampler(physical_gpu_index(local_rank))


def physical_gpu_index(local_rank: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        parts = [p for p in vis.split(",") if p.strip()]
        if local_rank < len(parts) and parts[local_rank].strip().isdigit():
            return int(parts[local_rank])
    return local_rank


# ---------------------------------------------------------------- our arm
class StepRunner:
    """Device buffers and the libispa call sequence of one chunk step."""

    def __init__(self, wl, device, seed=0):
        import torch

        from paper_2607_00712_gb300 import abi, synth
        from paper_2607_00712_gb300.device import LS, Ring, Window, bf16_tensor
        self.abi, self.torch = abi, torch
        H, d, P, L, F, Wn, nq, D = (wl[k] for k in ("H", "d", "P", "L", "F", "W", "nq", "D"))
        self.wl = wl
        self.win = Window(0, Wn)
        # three layers: F-layer (18-frame ring), L-layer (window ring), warmup layer (18-frame ring)
        self.rings = [Ring(H, d, P, F, 0, device), Ring(H, d, P, Wn, 0, device), Ring(H, d, P, F, 0, device)]
        self.inputs = []
        self.debug = False
        for li, ring in enumerate(self.rings):
            t0 = time.perf_counter()
            s = synth.make_step(seed * 100 + li, ring.c.capacity_frames, P, H, d, L)
            log(f"[bench] inputs of layer {li} drawn in {time.perf_counter() - t0:.1f} s")
            for f0 in range(0, ring.c.capacity_frames, L):
                n = min(L, ring.c.capacity_frames - f0)
                abi.ispa_kv_append(ring.c, bf16_tensor(s.k_hist[f0 * P:(f0 + n) * P], device),
                                   bf16_tensor(s.v_hist[f0 * P:(f0 + n) * P], device), n)
            self.inputs.append((bf16_tensor(s.q, device), bf16_tensor(s.k_cur, device), bf16_tensor(s.v_cur, device)))
        bf = torch.bfloat16
        self.out_full = torch.empty(nq, D, dtype=bf, device=device)
        self.out_local = torch.empty(nq, D, dtype=bf, device=device)
        self.a_full = torch.empty(nq, D, dtype=bf, device=device)
        self.a_loc = torch.empty(nq, D, dtype=bf, device=device)
        self.disc = torch.empty(nq, dtype=torch.float32, device=device)
        self.disc_sum = torch.zeros(1, dtype=torch.float32, device=device)
        self.dual_wsb = abi.ispa_attn_dual_workspace_size(H, nq)
        self.dual_ws = torch.empty(self.dual_wsb, dtype=torch.uint8, device=device)
        self.ls = LS(D, device)
        self.ls_wsb = abi.ispa_ls_accumulate_workspace_size(D, nq)
        self.ls_ws = torch.empty(self.ls_wsb, dtype=torch.uint8, device=device)
        self.ring_arr = (abi.KVRing * 3)()
        self.stream = torch.cuda.current_stream(device)
        self.launches_per_step = 8   # 3 attention + disc reduce + amax + convert + gram + append
        torch.cuda.synchronize(device)

    def outputs(self):
        """The step's result tensors (the ones an e2e run reads back)."""
        return [self.out_full, self.out_local, self.a_full, self.a_loc, self.disc]

    def step(self, ev=None, inputs=None, outs=None, in_events=None):
        """Enqueue one step; ev = list of 6 events to record between the calls (or None).

        inputs / outs: another set of (q, k_cur, v_cur) triples / result tensors of the same
        shapes (the e2e pipeline alternates two sets); default: the runner's own.
        in_events: one event per layer, recorded once that layer's inputs are on the device;
        the layer's attention call waits for its own (or None)."""
        abi, nq = self.abi, self.wl["nq"]
        s = self.stream
        inputs = self.inputs if inputs is None else inputs
        out_full, out_local, a_full, a_loc, disc = self.outputs() if outs is None else outs
        if self.debug:
            def rec(i):
                self.torch.cuda.synchronize()
                st, code = abi.ispa_last_device_error()
                log(f"[bench]   call {i} done, device status {st}/{code}")
        else:
            rec = (lambda i: ev[i].record(s)) if ev else (lambda i: None)
        wait_in = (lambda k: s.wait_event(in_events[k])) if in_events else (lambda k: None)
        rec(0)
        wait_in(0)
        q, kc, vc = inputs[0]
        abi.ispa_attn_full(self.rings[0].c, q, kc, vc, nq, 0.0, out_full, None, s)
        rec(1)
        wait_in(1)
        q, kc, vc = inputs[1]
        abi.ispa_attn_local(self.rings[1].c, self.win, q, kc, vc, nq, 0.0, out_local, None, s)
        rec(2)
        wait_in(2)
        q, kc, vc = inputs[2]
        abi.ispa_attn_dual(self.rings[2].c, self.win, q, kc, vc, nq, 0.0, a_full, a_loc, disc,
                           self.disc_sum, None, None, self.dual_ws, self.dual_wsb, s)
        rec(3)
        abi.ispa_ls_accumulate(self.ls.c, a_loc, a_full, nq, self.ls_ws, self.ls_wsb, s)
        rec(4)
        for i in range(3):
            self.ring_arr[i] = self.rings[i].c
        abi.ispa_kv_append_layers(self.ring_arr, [x[1] for x in inputs], [x[2] for x in inputs],
                                  self.wl["L"], s)
        for i in range(3):
            self.rings[i].c.frames_written = self.ring_arr[i].frames_written
        rec(5)


def timed_steps(r, steps, device, flush, rank, world, local_rank):
    """Time `steps` chunk steps of runner r: CUDA events between the calls of every step, L2
    flushed before each step outside its events, a barrier and a device synchronisation on
    both sides, clocks sampled inside the region.  Returns (segment ms [steps, 5], wall s,
    clocks); a region whose clocks the timing rules reject is measured once more."""
    import torch
    abi = r.abi
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(steps)]

    def once():
        sampler = make_sampler(local_rank) if rank == 0 else None
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(device)
        if sampler:
            sampler.start()
            time.sleep(0.05)
        t0 = time.perf_counter()
        for k in range(steps):
            flush.fill_(float(k))          # L2 flush, outside the step's events
            r.step(evs[k])
        torch.cuda.synchronize(device)
        t1 = time.perf_counter()
        if world > 1:
            torch.distributed.barrier()
        clocks = sampler.stop(t0, t1) if sampler else None
        st, code = abi.ispa_last_device_error()
        if st != abi.ISPA_OK:
            raise RuntimeError(f"device error in timed region: {code}")
        return t1 - t0, clocks

    wall, clocks = once()
    # A timed region that saw a hardware or thermal slowdown, or SM clocks well below their
    # maximum with no reason given (a clock lock left by someone else), is measured once more.
    again = int(clock_rejected(clocks))
    if world > 1:
        t = torch.tensor([again], device=device)
        torch.distributed.broadcast(t, 0)
        again = int(t.item())
    if again:
        log(f"[bench] clocks {clocks}: measuring the timed region once more")
        first = clocks
        wall, clocks = once()
        if clocks is not None:
            clocks = dict(clocks, remeasured=True, first_attempt=first)
    seg = np.array([[evs[k][i].elapsed_time(evs[k][i + 1]) for i in range(5)] for k in range(steps)])
    return seg, wall, clocks


def modes_of(seg, wl, pk):
    """Per-call means of the timed steps with their rates: attention TFLOP/s (and fraction of the
    measured dense bf16 peak), LS accumulate method-work and tile-work TFLOP/s, append GB/s."""
    mean = seg.mean(axis=0)
    ls_method, ls_tile = ls_flops(wl["D"], wl["nq"])
    app_bytes = 3 * 2 * 2 * wl["nq"] * wl["D"] * 2

    def attn(ms, fl, nk):
        tf = fl / (ms * 1e-3) / 1e12
        return dict(ms=ms, tflops=tf, frac=tf / pk["bf16"], nk=nk)

    modes = dict(
        full=attn(mean[0], wl["flops_full"], wl["nk_full"]),
        local=attn(mean[1], wl["flops_local"], wl["nk_local"]),
        dual=attn(mean[2], wl["flops_dual"], wl["nk_full"]),
        ls_accumulate=dict(ms=mean[3], method_gflop=ls_method / 1e9,
                           method_tflops=ls_method / (mean[3] * 1e-3) / 1e12,
                           method_frac=ls_method / (mean[3] * 1e-3) / 1e12 / pk["bf16"],
                           tile_tflops=ls_tile / (mean[3] * 1e-3) / 1e12),
        kv_append=dict(ms=mean[4], gbs=app_bytes / (mean[4] * 1e-3) / 1e9,
                       frac=app_bytes / (mean[4] * 1e-3) / 1e9 / pk["hbm"]),
    )
    for m in modes.values():
        for k_, v_ in list(m.items()):
            if isinstance(v_, float):
                m[k_] = round(v_, 4)
    return modes


def run_ours(args, rank, world, local_rank):
    import torch
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    from paper_2607_00712_gb300 import abi
    from paper_2607_00712_gb300.build import build_library
    t_start = time.perf_counter()
    build_library()
    abi.lib()
    wl = workload(args.model)
    pk = peaks()
    r = StepRunner(wl, device)
    log(f"[bench] set-up done in {time.perf_counter() - t_start:.1f} s")
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=device)

    for i in range(args.warmup):
        r.debug = i == 0
        r.step()
        r.debug = False
        torch.cuda.synchronize(device)
        log(f"[bench] warmup step {i} done at {time.perf_counter() - t_start:.1f} s")
    st, code = abi.ispa_last_device_error()
    if st != abi.ISPA_OK:
        raise RuntimeError(f"device error after warmup: {code}")

    seg, wall, clocks = timed_steps(r, args.steps, device, flush, rank, world, local_rank)
    step_ms = seg.sum(axis=1)
    total_ms = float(step_ms.sum())
    if world > 1:
        t = torch.tensor([total_ms], device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        total_ms = float(t.item())
    flops_step = wl["flops_full"] + wl["flops_local"] + wl["flops_dual"]
    ms_per_step = total_ms / args.steps
    value = world * flops_step / (ms_per_step * 1e-3) / 1e12
    modes = modes_of(seg, wl, pk)
    roofline = roofline_entry(args.model, modes["full"]["tflops"], pk)
    # the F-layer's tensor work per SM clock: independent of the clock the peak was measured at
    if clocks and clocks.get("sm_mhz"):
        roofline["flop_per_sm_cycle"] = round(wl["flops_full"] / (modes["full"]["ms"] * 1e-3) /
                                              (clocks["sm_mhz"] * 1e6) / torch.cuda.get_device_properties(
                                                  device).multi_processor_count, 1)

    log(f"[bench] timed steps done at {time.perf_counter() - t_start:.1f} s")
    extras = run_extras(r, wl, device)
    log(f"[bench] extras done at {time.perf_counter() - t_start:.1f} s")
    if args.configs:
        extras["rollout"] = run_rollout(wl, device, MODEL_LAYERS[args.model])
        extras["warmup_to_transition"] = run_warmup(wl, device)
        log(f"[bench] rollout and warmup configs done at {time.perf_counter() - t_start:.1f} s")
    e2e = run_e2e(r, args, device, flops_step, world)
    log(f"[bench] e2e done at {time.perf_counter() - t_start:.1f} s")
    launches_per_step = r.launches_per_step
    del r
    torch.cuda.empty_cache()

    shapes = {}
    for other in args.shapes:
        if other == args.model:
            continue
        shapes[other] = run_shape(other, args, device, flush, rank, world, local_rank, pk)
        log(f"[bench] {other} shape done at {time.perf_counter() - t_start:.1f} s")

    result = dict(metric=METRIC, value=round(value, 3), unit=UNIT, n_gpus=world, steps=args.steps,
                  warmup=args.warmup, ms_per_step=round(ms_per_step, 4), higher_is_better=True,
                  scaling="weak", vs_baseline=None, dtype="bf16", data="synthetic",
                  config=dict(workload=f"ISPA chunk step, {args.model}-shaped layer stack (F + L + dual + LS + append)",
                              heads=wl["H"], head_dim=wl["d"], tokens_per_frame=wl["P"], n_q=wl["nq"],
                              f_ring_frames=wl["F"], window_frames=wl["W"], parallelism=f"replicas x{world}",
                              l2="flushed between steps (256 MB write outside timed events)"),
                  modes=modes, roofline=roofline, e2e=e2e, shapes=shapes, extras=extras,
                  gpu_launches=launches_per_step * args.steps, clocks=clocks,
                  wall_s=round(wall, 3))
    if rank == 0:
        if args.cpu_baseline:
            result["cpu_baseline"] = cpu_baseline(wl, args.cpu_sample_rows)
        print(json.dumps(result), flush=True)


def run_shape(model, args, device, flush, rank, world, local_rank, pk):
    """The same chunk step at another model shape, measured exactly like the headline one (same
    steps, L2 flushed outside the events, clocks sampled), with its own roofline entry and, unless
    --no-configs, that shape's rollout and warmup-to-transition workloads."""
    import torch
    wl = workload(model)
    r = StepRunner(wl, device, seed=1)
    for _ in range(args.warmup):
        r.step()
    torch.cuda.synchronize(device)
    seg, wall, clocks = timed_steps(r, args.steps, device, flush, rank, world, local_rank)
    ms = float(seg.sum(axis=1).mean())
    flops_step = wl["flops_full"] + wl["flops_local"] + wl["flops_dual"]
    modes = modes_of(seg, wl, pk)
    out = dict(workload=f"ISPA chunk step, {model}-shaped layer stack (F + L + dual + LS + append)",
               heads=wl["H"], head_dim=wl["d"], n_q=wl["nq"], value=round(flops_step / (ms * 1e-3) / 1e12, 3),
               unit=UNIT, ms_per_step=round(ms, 4), steps=args.steps, modes=modes,
               roofline=roofline_entry(model, modes["full"]["tflops"], pk), clocks=clocks)
    del r
    torch.cuda.empty_cache()
    if args.configs:
        out["rollout"] = run_rollout(wl, device, MODEL_LAYERS[model])
        torch.cuda.empty_cache()
        out["warmup_to_transition"] = run_warmup(wl, device)
        torch.cuda.empty_cache()
    return out


def run_extras(r, wl, device, reps=20):
    """Once-per-run figures outside the step: the paper's two-call dual pass (Eq. 9-12: local
    branch, history branch, LSE merge) against the fused one-sweep dual kernel, and the
    closed-form solve (Eq. 5-6) of the accumulated state."""
    import torch
    abi = r.abi
    nq, H, d, D = wl["nq"], wl["H"], wl["d"], wl["D"]
    q, kc, vc = r.inputs[2]
    ring = r.rings[2].c
    o_loc = torch.empty(nq, D, dtype=torch.bfloat16, device=device)
    o_hist = torch.empty_like(o_loc)
    fused = torch.empty_like(o_loc)
    l_loc = torch.empty(H, nq, dtype=torch.float32, device=device)
    l_hist = torch.empty_like(l_loc)
    l_out = torch.empty_like(l_loc)
    s = r.stream
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    t_loc = t_hist = t_merge = t_dual = 0.0
    for _ in range(reps):
        ev[0].record(s)
        abi.ispa_attn_local(ring, r.win, q, kc, vc, nq, 0.0, o_loc, l_loc, s)
        ev[1].record(s)
        abi.ispa_attn_hist(ring, r.win, q, nq, 0.0, o_hist, l_hist, s)
        ev[2].record(s)
        abi.ispa_lse_merge(o_loc, l_loc, o_hist, l_hist, nq, H, d, fused, l_out, s)
        ev[3].record(s)
        abi.ispa_attn_dual(ring, r.win, q, kc, vc, nq, 0.0, r.a_full, r.a_loc, r.disc, r.disc_sum, None, None,
                           r.dual_ws, r.dual_wsb, s)
        ev[4].record(s)
        torch.cuda.synchronize(device)
        t_loc += ev[0].elapsed_time(ev[1])
        t_hist += ev[1].elapsed_time(ev[2])
        t_merge += ev[2].elapsed_time(ev[3])
        t_dual += ev[3].elapsed_time(ev[4])
    dec = (t_loc + t_hist + t_merge) / reps
    out = dict(decomposed_dual_ms=round(dec, 4), fused_dual_ms=round(t_dual / reps, 4),
               decomposed_merge_ms=round(t_merge / reps, 4),
               merge_share_of_decomposed=round(t_merge / reps / dec, 4))
    # the decomposed pass's discrepancy from its two stored outputs (HBM-bound: both bf16
    # [n_q][D] outputs read once, disc written), L2 flushed before every repetition
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    disc = torch.empty(nq, dtype=torch.float32, device=device)
    dsum = torch.zeros(1, dtype=torch.float32, device=device)
    t_disc = 0.0
    for i in range(reps + 3):
        flush.fill_(float(i))
        ev[0].record(s)
        abi.ispa_discrepancy(fused, o_loc, nq, D, disc, dsum, s)
        ev[1].record(s)
        torch.cuda.synchronize(device)
        if i >= 3:
            t_disc += ev[0].elapsed_time(ev[1])
    t_disc /= reps
    # LS accumulate in its exact form (Delta as a bf16 hi / lo pair) against the default scaled
    # form on the same inputs, L2 flushed before each
    ev6 = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    t_ls = np.zeros(2)
    for i in range(reps + 3):
        flush.fill_(float(i))
        ev6[0].record(s)
        abi.ispa_ls_accumulate(r.ls.c, r.a_loc, r.a_full, nq, r.ls_ws, r.ls_wsb, s)
        ev6[1].record(s)
        flush.fill_(float(i) + 0.5)
        ev6[2].record(s)
        abi.ispa_ls_accumulate_ex(r.ls.c, r.a_loc, r.a_full, nq, abi.ISPA_LS_EXACT_DELTA, r.ls_ws, r.ls_wsb, s)
        ev6[3].record(s)
        torch.cuda.synchronize(device)
        if i >= 3:
            t_ls += [ev6[0].elapsed_time(ev6[1]), ev6[2].elapsed_time(ev6[3])]
    t_ls /= reps
    _, tile_exact = ls_flops(D, nq, exact=True)
    out.update(ls_accumulate_scaled_ms=round(t_ls[0], 4), ls_accumulate_exact_ms=round(t_ls[1], 4),
               ls_exact_tile_tflops=round(tile_exact / (t_ls[1] * 1e-3) / 1e12, 1))
    disc_bytes = 2 * nq * D * 2 + nq * 4
    pk = peaks()
    out.update(discrepancy_ms=round(t_disc, 4), discrepancy_gbs=round(disc_bytes / (t_disc * 1e-3) / 1e9, 1),
               discrepancy_frac_of_hbm=round(disc_bytes / (t_disc * 1e-3) / 1e9 / pk["hbm"], 4),
               discrepancy_bytes=disc_bytes)
    del flush
    # closed-form solve of the accumulated state (once per transition)
    from paper_2607_00712_gb300 import synth
    W = torch.from_numpy(synth.make_weight(1, D, D)).to(device)
    dW = torch.empty(D, D, dtype=torch.float32, device=device)
    wsb = abi.ispa_ls_solve_workspace_size(D, D)
    ws = torch.empty(wsb, dtype=torch.uint8, device=device)
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    try:
        abi.ispa_ls_solve(r.ls.c, W, D, 1e-3, dW, ws, wsb, s)
        out["ls_solve_ms"] = round((time.perf_counter() - t0) * 1e3, 2)
        out["ls_solve_dim"] = D
    except abi.IspaError as e:
        out["ls_solve_error"] = str(e)
        dW.zero_()
    out.update(run_w8a8(r, wl, device, W, dW, reps))
    out.update(run_qk8(r, wl, device, reps))
    out.update(run_kv8(r, wl, device, reps))
    return out


def run_qk8(r, wl, device, reps, seed=0):
    """The F-layer attention with 8-bit queries and keys (e4m3 Q K^T, bf16 P V) on the same
    history as the step's F-layer ring: the ring's per-head key scales come from quantising the
    history once; per step the chunk's queries are quantised per 128-token block and its keys
    with the ring's scales (timed separately).  L2 is flushed
    before every repetition, as in the step."""
    import torch
    from paper_2607_00712_gb300 import synth
    from paper_2607_00712_gb300.device import Ring, bf16_tensor
    abi = r.abi
    H, d, P, L, F, nq = (wl[k] for k in ("H", "d", "P", "L", "F", "nq"))
    if d != 128:
        return {}
    s = synth.make_step(seed * 100 + 0, F, P, H, d, L)          # the F-layer ring's inputs
    kh = bf16_tensor(s.k_hist, device)
    vh = bf16_tensor(s.v_hist, device)
    n_hist = kh.shape[0]
    k_hist_codes = torch.empty(n_hist, H, d, dtype=torch.uint8, device=device)
    k_ring_scale = torch.empty(H, dtype=torch.float32, device=device)
    abi.ispa_quantize_heads_e4m3(kh, n_hist, H, d, k_hist_codes, k_ring_scale)
    ring = Ring(H, d, P, F, 0, device, k_e4m3=True)
    for f0 in range(0, F, L):
        n = min(L, F - f0)
        abi.ispa_kv_append_qk8(ring.c, kh[f0 * P:(f0 + n) * P], vh[f0 * P:(f0 + n) * P], n, k_ring_scale)
    q, kc, vc = r.inputs[0]
    q8 = torch.empty(nq, H, d, dtype=torch.uint8, device=device)
    k8 = torch.empty_like(q8)
    qs = torch.empty(H, (nq + 127) // 128, dtype=torch.float32, device=device)
    out = torch.empty(nq, H * d, dtype=torch.bfloat16, device=device)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    st = r.stream
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    t_q = t_a = 0.0
    for i in range(reps + 3):
        flush.fill_(float(i))
        ev[0].record(st)
        abi.ispa_quantize_q_e4m3(q, nq, H, d, q8, qs, st)
        abi.ispa_quantize_k_e4m3(kc, nq, H, d, k_ring_scale, k8, st)
        ev[1].record(st)
        abi.ispa_attn_full_qk8(ring.c, k_ring_scale, q8, qs, k8, k_ring_scale, vc, nq, 0.0, out, None, st)
        ev[2].record(st)
        torch.cuda.synchronize(device)
        if i >= 3:
            t_q += ev[0].elapsed_time(ev[1])
            t_a += ev[1].elapsed_time(ev[2])
    t_q, t_a = t_q / reps, t_a / reps
    tf = wl["flops_full"] / (t_a * 1e-3) / 1e12
    return dict(qk8_full_ms=round(t_a, 4), qk8_full_tflops=round(tf, 1),
                qk8_chunk_quant_ms=round(t_q, 4), qk8_nk=F * P + nq)


def run_kv8(r, wl, device, reps, seed=0):
    """The F-layer attention with 8-bit Q K^T and 8-bit P V (e4m3 keys and d-major e4m3 values in
    the ring, e4m3 probabilities in the kernel) on the same history as the step's F-layer ring;
    per step the chunk's queries, keys and values are quantised (timed separately).  L2 is
    flushed before every repetition."""
    import torch
    from paper_2607_00712_gb300 import synth
    from paper_2607_00712_gb300.device import Ring, bf16_tensor
    abi = r.abi
    H, d, P, L, F, nq = (wl[k] for k in ("H", "d", "P", "L", "F", "nq"))
    if d != 128 or P % 4:
        return {}
    s = synth.make_step(seed * 100 + 0, F, P, H, d, L)          # the F-layer ring's inputs
    kh = bf16_tensor(s.k_hist, device)
    vh = bf16_tensor(s.v_hist, device)
    n_hist = kh.shape[0]
    scratch = torch.empty(n_hist, H, d, dtype=torch.uint8, device=device)
    k_scale = torch.empty(H, dtype=torch.float32, device=device)
    v_scale = torch.empty(H, dtype=torch.float32, device=device)
    abi.ispa_quantize_heads_e4m3(kh, n_hist, H, d, scratch, k_scale)
    abi.ispa_quantize_heads_e4m3(vh, n_hist, H, d, scratch, v_scale)
    ring = Ring(H, d, P, F, 0, device, kv_e4m3=True)
    for f0 in range(0, F, L):
        n = min(L, F - f0)
        abi.ispa_kv_append_kv8(ring.c, kh[f0 * P:(f0 + n) * P], vh[f0 * P:(f0 + n) * P], n, k_scale, v_scale)
    del scratch, kh, vh
    q, kc, vc = r.inputs[0]
    q8 = torch.empty(nq, H, d, dtype=torch.uint8, device=device)
    k8 = torch.empty_like(q8)
    qs = torch.empty(H, (nq + 127) // 128, dtype=torch.float32, device=device)
    ld = (nq + 15) // 16 * 16
    vt8 = torch.empty(H, d, ld, dtype=torch.uint8, device=device)
    out = torch.empty(nq, H * d, dtype=torch.bfloat16, device=device)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=device)
    st = r.stream
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    t_q = t_a = 0.0
    for i in range(reps + 3):
        flush.fill_(float(i))
        ev[0].record(st)
        abi.ispa_quantize_q_e4m3(q, nq, H, d, q8, qs, st)
        abi.ispa_quantize_k_e4m3(kc, nq, H, d, k_scale, k8, st)
        abi.ispa_quantize_vt_e4m3(vc, nq, H, d, v_scale, vt8, ld, st)
        ev[1].record(st)
        abi.ispa_attn_full_kv8(ring.c, k_scale, v_scale, q8, qs, k8, k_scale, vt8, ld, nq, 0.0, out, None, st)
        ev[2].record(st)
        torch.cuda.synchronize(device)
        if i >= 3:
            t_q += ev[0].elapsed_time(ev[1])
            t_a += ev[1].elapsed_time(ev[2])
    t_q, t_a = t_q / reps, t_a / reps
    tf = wl["flops_full"] / (t_a * 1e-3) / 1e12
    return dict(kv8_full_ms=round(t_a, 4), kv8_full_tflops=round(tf, 1), kv8_chunk_quant_ms=round(t_q, 4),
                kv8_ring_bytes=int(abi.ispa_ring_bytes(ring.c)))


def run_w8a8(r, wl, device, W, dW, reps):
    """The attention output projection with 8-bit weights and activations (Sec. 4) on the
    injected weight W + dW: weight quantisation (once per transition), then per step the
    activation quantisation and the e4m3 GEMM, next to a cuBLAS bf16 GEMM of the same shape
    (context for the latency breakdown).  Inputs stay L2-warm across the repetitions."""
    import torch
    abi = r.abi
    T, D = wl["nq"], wl["D"]
    a = r.a_full                                   # [T][D] bf16, a real attention output
    wq = torch.empty(D, D, dtype=torch.uint8, device=device)
    ws = torch.empty(D, dtype=torch.float32, device=device)
    aq = torch.empty(T, D, dtype=torch.uint8, device=device)
    sa = torch.empty(T, dtype=torch.float32, device=device)
    y = torch.empty(T, D, dtype=torch.bfloat16, device=device)
    s = r.stream
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    ev[0].record(s)
    abi.ispa_quantize_weight_e4m3(W, dW, D, D, wq, ws, s)
    ev[1].record(s)
    torch.cuda.synchronize(device)
    t_wq = ev[0].elapsed_time(ev[1])
    w_bf16 = (W + dW).to(torch.bfloat16)
    t_q = t_mm = t_ref = 0.0
    for i in range(reps + 3):
        ev[0].record(s)
        abi.ispa_quantize_rows_e4m3(a, T, D, aq, sa, s)
        ev[1].record(s)
        abi.ispa_linear_w8a8(aq, sa, wq, ws, T, D, D, y, s)
        ev[2].record(s)
        torch.matmul(a, w_bf16)
        ev[3].record(s)
        torch.cuda.synchronize(device)
        if i >= 3:
            t_q += ev[0].elapsed_time(ev[1])
            t_mm += ev[1].elapsed_time(ev[2])
            t_ref += ev[2].elapsed_time(ev[3])
    t_q, t_mm, t_ref = t_q / reps, t_mm / reps, t_ref / reps
    flops = 2.0 * T * D * D
    pk = peaks()
    fp8_peak = 2.0 * pk["bf16"]                    # measured bf16 peak x the nominal fp8 / bf16 ratio
    tf = flops / (t_mm * 1e-3) / 1e12
    return dict(w8a8_weight_quant_ms=round(t_wq, 4), w8a8_act_quant_ms=round(t_q, 4),
                w8a8_gemm_ms=round(t_mm, 4), w8a8_gemm_tflops=round(tf, 1),
                w8a8_gemm_frac_of_fp8_peak=round(tf / fp8_peak, 4), w8a8_fp8_peak_tflops=fp8_peak,
                cublas_bf16_projection_ms=round(t_ref, 4),
                w8a8_shape=f"{T} x {D} -> {D}")


def _device_qkv(g, n_frames, P, H, d):
    """One layer's chunk q, k, v drawn on the device with the synthetic recipe of the parity
    inputs: N(0, 1) entries, every key of a frame and head shifted by an offset vector
    ~ N(0, 0.5^2), rounded to bf16."""
    import torch
    dev = g.device
    q = torch.randn(n_frames * P, H, d, device=dev, generator=g)
    k = torch.randn(n_frames, P, H, d, device=dev, generator=g)
    k += 0.5 * torch.randn(n_frames, 1, H, d, device=dev, generator=g)
    v = torch.randn(n_frames * P, H, d, device=dev, generator=g)
    return tuple(x.reshape(n_frames * P, H, d).to(torch.bfloat16) for x in (q, k, v))


def run_rollout(wl, device, n_layers, steps=20):
    """The AR rollout workload: `steps` chunk steps of `n_layers` blocks alternating F-layers
    (attention over every past frame; the cache grows from 0 to 3 * (steps - 1) frames, up to
    93,600 keys) and L-layers (chunk + 6-frame window), each step ending with the batched KV
    append of all layers.  Every layer has its own ring and its own chunk q, k, v (drawn on the
    device before each step, outside the timed events); L2 is not flushed between layers.
    The rollout's keys (the F-rings hold up to 60 frames) keep the working set far above L2."""
    import torch
    from paper_2607_00712_gb300 import abi
    from paper_2607_00712_gb300.device import Ring, Window
    H, d, P, L, Wn, nq = (wl[k] for k in ("H", "d", "P", "L", "W", "nq"))
    cap_f = L * steps
    rings = [Ring(H, d, P, cap_f if li % 2 == 0 else Wn, 0, device) for li in range(n_layers)]
    win = Window(0, Wn)
    outs = torch.empty(nq, H * d, dtype=torch.bfloat16, device=device)
    arr = (abi.KVRing * n_layers)()
    s = torch.cuda.current_stream(device)
    e0, ea, e1 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
    g = torch.Generator(device=device)
    g.manual_seed(7)
    total_ms, append_ms, flops, step_ms = 0.0, 0.0, 0.0, []
    for step in range(steps):
        past = L * step
        chunk = [_device_qkv(g, L, P, H, d) for _ in range(n_layers)]
        torch.cuda.synchronize(device)
        e0.record(s)
        for li in range(n_layers):
            q, kc, vc = chunk[li]
            if li % 2 == 0:
                abi.ispa_attn_full(rings[li].c, q, kc, vc, nq, 0.0, outs, None, s)
                flops += attn_flops(nq, past * P + nq, d, H)
            else:
                abi.ispa_attn_local(rings[li].c, win, q, kc, vc, nq, 0.0, outs, None, s)
                flops += attn_flops(nq, min(past, Wn) * P + nq, d, H)
        for li in range(n_layers):
            arr[li] = rings[li].c
        ea.record(s)
        abi.ispa_kv_append_layers(arr, [c[1] for c in chunk], [c[2] for c in chunk], L, s)
        for li in range(n_layers):
            rings[li].c.frames_written = arr[li].frames_written
        e1.record(s)
        torch.cuda.synchronize(device)
        step_ms.append(e0.elapsed_time(e1))
        total_ms += step_ms[-1]
        append_ms += ea.elapsed_time(e1)
        if step < steps - 1:
            del chunk
    # the append alone: one batched launch over all layers against one launch per layer
    # (the rings are full here, so every append evicts the oldest frames)
    app_bytes = n_layers * 2 * 2 * nq * H * d * 2
    reps = 5
    torch.cuda.synchronize(device)
    e0.record(s)
    for _ in range(reps):
        for li in range(n_layers):
            arr[li] = rings[li].c
        abi.ispa_kv_append_layers(arr, [c[1] for c in chunk], [c[2] for c in chunk], L, s)
        for li in range(n_layers):
            rings[li].c.frames_written = arr[li].frames_written
    e1.record(s)
    torch.cuda.synchronize(device)
    batched = e0.elapsed_time(e1) / reps
    e0.record(s)
    for _ in range(reps):
        for li in range(n_layers):
            abi.ispa_kv_append(rings[li].c, chunk[li][1], chunk[li][2], L, s)
    e1.record(s)
    torch.cuda.synchronize(device)
    per_layer = e0.elapsed_time(e1) / reps
    return dict(layers=n_layers, steps=steps, max_keys=(L * (steps - 1)) * P + nq, ms=round(total_ms, 2),
                first_step_ms=round(step_ms[0], 3), last_step_ms=round(step_ms[-1], 3),
                attention_tflop=round(flops / 1e12, 2),
                attention_tflops=round(flops / ((total_ms - append_ms) * 1e-3) / 1e12, 1),
                append_ms_per_step=round(append_ms / steps, 4),
                append_all_layers=dict(batched_ms=round(batched, 4), per_layer_calls_ms=round(per_layer, 4),
                                       batched_gbs=round(app_bytes / (batched * 1e-3) / 1e9, 0),
                                       per_layer_gbs=round(app_bytes / (per_layer * 1e-3) / 1e9, 0)))


def run_warmup(wl, device, steps=8, cache_frames=24):
    """The warmup-to-transition workload: `steps` dual passes (full set = a 24-frame cache +
    the chunk, local = chunk + 6-frame window) with the discrepancy reduction and the LS
    accumulation of every step's A_loc / A_full, then the closed-form solve once."""
    import torch
    from paper_2607_00712_gb300 import abi, synth
    from paper_2607_00712_gb300.device import LS, Ring, Window
    H, d, P, L, Wn, nq, D = (wl[k] for k in ("H", "d", "P", "L", "W", "nq", "D"))
    g = torch.Generator(device=device)
    g.manual_seed(11)
    ring = Ring(H, d, P, cache_frames, 0, device)
    for f0 in range(0, cache_frames, L):
        _, kk, vv = _device_qkv(g, L, P, H, d)
        abi.ispa_kv_append(ring.c, kk, vv, L)
    win = Window(0, Wn)
    st = LS(D, device)
    a_full = torch.empty(nq, D, dtype=torch.bfloat16, device=device)
    a_loc = torch.empty_like(a_full)
    disc = torch.empty(nq, dtype=torch.float32, device=device)
    dsum = torch.zeros(1, dtype=torch.float32, device=device)
    wsb = abi.ispa_attn_dual_workspace_size(H, nq)
    ws = torch.empty(wsb, dtype=torch.uint8, device=device)
    lwsb = abi.ispa_ls_accumulate_workspace_size(D, nq)
    lws = torch.empty(lwsb, dtype=torch.uint8, device=device)
    qkv = [_device_qkv(g, L, P, H, d) for _ in range(steps)]
    s = torch.cuda.current_stream(device)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    t_dual = t_ls = 0.0
    torch.cuda.synchronize(device)
    for q, kc, vc in qkv:
        ev[0].record(s)
        abi.ispa_attn_dual(ring.c, win, q, kc, vc, nq, 0.0, a_full, a_loc, disc, dsum, None, None, ws, wsb, s)
        ev[1].record(s)
        abi.ispa_ls_accumulate(st.c, a_loc, a_full, nq, lws, lwsb, s)
        ev[2].record(s)
        torch.cuda.synchronize(device)
        t_dual += ev[0].elapsed_time(ev[1])
        t_ls += ev[1].elapsed_time(ev[2])
    W = torch.from_numpy(synth.make_weight(3, D, D)).to(device)
    dW = torch.empty(D, D, dtype=torch.float32, device=device)
    swsb = abi.ispa_ls_solve_workspace_size(D, D)
    sws = torch.empty(swsb, dtype=torch.uint8, device=device)
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    nk = cache_frames * P + nq
    out = dict(steps=steps, keys_full=nk, dual_ms_per_step=round(t_dual / steps, 4),
               dual_tflops=round(attn_flops(nq, nk, d, H) / (t_dual / steps * 1e-3) / 1e12, 1),
               ls_accumulate_ms_per_step=round(t_ls / steps, 4), tokens=steps * nq,
               disc_sq_sum=float(dsum.item()))
    try:
        out["eps"] = abi.ispa_ls_solve(st.c, W, D, 1e-3, dW, sws, swsb, s)
        out["solve_ms"] = round((time.perf_counter() - t0) * 1e3, 2)
    except abi.IspaError as e:
        out["solve_error"] = str(e)
    return out


def run_e2e(r, args, device, flops_step, world):
    """The same step through the C-ABI with pinned host inputs / outputs copied inside the timed region.

    Every step copies its own inputs host->device before its compute and reads its results
    device->host after it.  The copies of step i+1 (in) and i-1 (out) run on two copy streams
    while step i computes: two sets of device inputs and outputs alternate, ordered by events
    (each layer's call waits for that layer's inputs, each result is read back once the call
    that writes it has finished; a set is refilled only after the step that used it has finished
    computing and has been read back).  Timed from the first copy in to the last copy out,
    divided by the number of steps.
    """
    import torch
    host_in = [[t.cpu().pin_memory() for t in trip] for trip in r.inputs]
    dev_in = [r.inputs, [tuple(torch.empty_like(t) for t in trip) for trip in r.inputs]]
    dev_out = [r.outputs(), [torch.empty_like(t) for t in r.outputs()]]
    host_out = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in r.outputs()]
    h2d = sum(t.numel() * t.element_size() for trip in host_in for t in trip)
    d2h = sum(t.numel() * t.element_size() for t in host_out)
    s_comp = r.stream
    s_in, s_out = torch.cuda.Stream(device), torch.cuda.Stream(device)
    n = max(3, min(args.steps, 20))

    def run(steps, e_start=None, e_end=None):
        ev_comp, ev_out = [], []
        for i in range(steps):
            b = i % 2
            e_in = []
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(ev_comp[i - 2])          # set b no longer read by step i-2
                if i == 0 and e_start is not None:
                    e_start.record(s_in)
                for trip_h, trip_d in zip(host_in, dev_in[b]):
                    for h, dv in zip(trip_h, trip_d):
                        dv.copy_(h, non_blocking=True)
                    e = torch.cuda.Event()
                    e.record(s_in)                           # this layer's inputs are in
                    e_in.append(e)
            if i >= 2:
                s_comp.wait_event(ev_out[i - 2])             # outputs of set b read back
            ev = [torch.cuda.Event() for _ in range(6)]
            r.step(ev=ev, inputs=dev_in[b], outs=dev_out[b], in_events=e_in)
            ev_comp.append(ev[5])
            with torch.cuda.stream(s_out):
                # out_full after the F call, out_local after L, a_full, a_loc, disc after the dual
                for h, dv, k in zip(host_out, dev_out[b], (1, 2, 3, 3, 3)):
                    s_out.wait_event(ev[k])
                    h.copy_(dv, non_blocking=True)
                e_o = torch.cuda.Event()
                e_o.record(s_out)
                ev_out.append(e_o)
        if e_end is not None:
            e_end.record(s_out)

    run(2)
    torch.cuda.synchronize(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    run(n, e0, e1)
    torch.cuda.synchronize(device)
    ms = e0.elapsed_time(e1) / n
    return dict(value=round(world * flops_step / (ms * 1e-3) / 1e12, 3), unit=UNIT, h2d_bytes_per_step=h2d,
                d2h_bytes_per_step=d2h, ms_per_step=round(ms, 4), steps=n,
                overlap="copies on two streams, double-buffered device inputs and outputs")


# ---------------------------------------------------------------- oracle legs
def _oracle_sample(wl, rows_per_mode, seed=0):
    """Inputs of one bounded oracle sample: the three layers' steps, sampled query rows."""
    from paper_2607_00712_gb300 import synth
    H, d, P, L, F, Wn = (wl[k] for k in ("H", "d", "P", "L", "F", "W"))
    steps = [synth.make_step(seed * 100 + li, cap, P, H, d, L) for li, cap in enumerate([F, Wn, F])]
    rng = np.random.default_rng(seed)
    rows = np.sort(rng.choice(wl["nq"], rows_per_mode, replace=False))
    return steps, rows


def _oracle_step(wl, steps, rows):
    from oracle import attention as oat
    from oracle import ls as ols
    P, Wn = wl["P"], wl["W"]
    s0, s1, s2 = steps
    oat.attn_full(s0.q, s0.k_hist, s0.v_hist, s0.k_cur, s0.v_cur, P, rows=rows)
    oat.attn_local(s1.q, s1.k_hist, s1.v_hist, s1.k_cur, s1.v_cur, P, 0, Wn, rows=rows)
    r = oat.attn_dual(s2.q, s2.k_hist, s2.v_hist, s2.k_cur, s2.v_cur, P, 0, Wn, rows=rows)
    n = len(rows)
    st = ols.ls_state(wl["D"])
    ols.ls_accumulate(st, r["a_loc"].reshape(n, -1), r["a_full"].reshape(n, -1))
    # algorithmic attention FLOPs of the sampled rows (same count as the GPU metric)
    return (wl["flops_full"] + wl["flops_local"] + wl["flops_dual"]) * n / wl["nq"]


def cpu_baseline(wl, rows):
    steps, rs = _oracle_sample(wl, rows)
    t0 = time.perf_counter()
    flops = _oracle_step(wl, steps, rs)
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return dict(value=round(flops / dt / 1e12, 6), unit=UNIT, cores=cores, kind="oracle",
                sample=f"{rows} of {wl['nq']} query rows of each mode (full, local, dual) x all heads, "
                       f"plus LS accumulation of those rows; fp64 numpy, {dt:.1f} s",
                seconds=round(dt, 2), blas_threads=blas_threads())


def blas_threads():
    """Threads of numpy's BLAS as reported by threadpoolctl, else the environment's limit."""
    try:
        from threadpoolctl import threadpool_info
        n = [d.get("num_threads") for d in threadpool_info() if d.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:   # threadpoolctl is optional
        pass
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return "library default (threadpoolctl not installed)"


def run_reference(args, rank, world):
    if rank != 0:
        return
    wl = workload(args.model)
    rows = args.ref_rows
    steps, rs = _oracle_sample(wl, rows)
    for _ in range(args.warmup if args.warmup < 1 else 1):
        _oracle_step(wl, steps, rs[:8])
    t0 = time.perf_counter()
    flops = 0.0
    for _ in range(args.steps):
        flops += _oracle_step(wl, steps, rs)
    dt = time.perf_counter() - t0
    value = flops / dt / 1e12
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    res = dict(impl="reference", metric=METRIC, value=round(value, 6), unit=UNIT, n_gpus=world, steps=args.steps,
               warmup=args.warmup, ms_per_step=round(dt / args.steps * 1e3, 2), higher_is_better=True,
               scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
               config=dict(workload=f"ISPA chunk step, {args.model}-shaped layer stack (F + L + dual + LS)",
                           heads=wl["H"], head_dim=wl["d"], tokens_per_frame=wl["P"], n_q=wl["nq"],
                           sample_rows=rows),
               cpu_baseline=dict(value=round(value, 6), unit=UNIT, cores=cores, kind="oracle",
                                 sample=f"{rows} query rows per mode per step"),
               e2e=dict(value=round(value, 6), unit=UNIT, h2d_bytes_per_step=0, d2h_bytes_per_step=0))
    print(json.dumps(res), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--model", choices=sorted(MODELS), default="1.3b")
    ap.add_argument("--shapes", default="1.3b,14b",
                    help="model shapes measured after the headline one (comma list; the headline is --model)")
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--no-configs", dest="configs", action="store_false",
                    help="skip the rollout and warmup-to-transition workloads in the extras")
    ap.add_argument("--cpu-sample-rows", type=int, default=1536)
    ap.add_argument("--ref-rows", type=int, default=32)
    ap.add_argument("--watchdog", type=float, default=300.0, help="dump Python stacks after this many s")
    args = ap.parse_args()
    args.shapes = [x for x in args.shapes.split(",") if x]
    for x in args.shapes:
        if x not in MODELS:
            ap.error(f"unknown shape {x}")
    import faulthandler
    faulthandler.dump_traceback_later(args.watchdog, exit=False)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
