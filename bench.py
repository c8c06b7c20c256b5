"""Benchmark of the grouped ternary (W1.58A16) linear hot path on GB300.

One step = one pass of the whole path over one synthetic batch of the Mamba-2
1.3B in_proj prefill (W fp32 [8512, 2048], g = 128, X bf16 [16384, 2048],
dY bf16 [16384, 8512]): tq_quantize_with_transpose (absmean scale + ternary codes
+ packing, and the transposed codes that dX streams, in one launch), tq_linear_fwd
(Y = X W^T), and the STE backward dX = dY W^ and dW = dY^T X.
``value`` is the algorithmic TFLOP/s of the three GEMMs (3 x 2 M N K per step)
over the device time of the whole step, inputs already in HBM; ``e2e`` is the
same metric through the C ABI with pinned host buffers, host<->device copies of
every input and output inside the timed region.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun (N > 1) every rank runs its own replica of the step (weak
scaling, no collective on the data path); rank 0 prints the JSON line.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

IN_PROJ = (8512, 2048)
OUT_PROJ = (2048, 4096)
M_PREFILL = 16384  # batch 8 x seq 2048
G = 128
N_LAYERS = 48
METRIC = "W1.58A16 linear fwd+bwd TFLOP/s"
WORKLOAD = ("Mamba-2 1.3B in_proj prefill, one step = tq_quantize_with_transpose W[8512,2048] "
            "(g=128: codes, scales, zero counts and the transposed codes) + tq_linear_fwd + "
            "tq_linear_bwd (dX, dW) at M=16384 (batch 8 x seq 2048)")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ------------------------------------------------------------------ helpers
def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def kernel_hash(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2606_18114_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, files):
    """DRAM bytes per launch from a committed ncu capture, if the kernel is unchanged."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel)
    if not e or e.get("source_sha") != kernel_hash(files):
        return None
    return e.get("dram_bytes_per_launch")


class ClockSampler:
    """SM clock, power and clock-event reasons while the timed region runs.

    Polls NVML (the driver's libnvidia-ml, through ctypes) every ~2 ms from a
    thread; ``mark(True)`` / ``mark(False)`` bracket the timed region on the host
    (the launches are queued inside it and the final synchronise returns when the
    device is done), and only samples taken inside the bracket are reported.
    Falls back to ``nvidia-smi -lms 20`` when NVML cannot be loaded."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    # clock-event reason bits of NVML
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, gpu_index: int, period_s: float = 0.002):
        self.idx = gpu_index
        self.period = period_s
        self.proc = None
        self.thread = None
        self.samples = []      # (t, sm_mhz, power_w, reasons bitmask)
        self.window = [None, None]
        self.sm_max = None
        self.source = None

    def _nvml_handle(self):
        import ctypes
        lib = None
        for name in ("libnvidia-ml.so.1", "libnvidia-ml.so"):
            try:
                lib = ctypes.CDLL(name)
                break
            except OSError:
                continue
        if lib is None or lib.nvmlInit_v2() != 0:
            return None, None
        h = ctypes.c_void_p()
        uuid = None
        try:
            uuid = str(torch.cuda.get_device_properties(self.idx).uuid)
        except Exception:
            pass
        ok = False
        if uuid:
            for u in (uuid, "GPU-" + uuid):
                if lib.nvmlDeviceGetHandleByUUID(u.encode(), ctypes.byref(h)) == 0:
                    ok = True
                    break
        if not ok and lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(self.idx), ctypes.byref(h)) != 0:
            return None, None
        return lib, h

    def _poll(self, lib, h):
        import ctypes
        clk, pw, mx = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        get_reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
        if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
            self.sm_max = float(mx.value)
        while not self._stop:
            t = time.perf_counter()
            if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0:
                p = pw.value / 1000.0 if lib.nvmlDeviceGetPowerUsage(h, ctypes.byref(pw)) == 0 else None
                r = rs.value if get_reasons(h, ctypes.byref(rs)) == 0 else 0
                self.samples.append((t, float(clk.value), p, int(r)))
            time.sleep(self.period)

    def mark(self, start: bool):
        self.window[0 if start else 1] = time.perf_counter()

    def __enter__(self):
        import threading
        self._stop = False
        lib, h = (None, None)
        try:
            lib, h = self._nvml_handle()
        except Exception:
            lib = None
        if lib is not None:
            self.source = "nvml, 2 ms"
            self.thread = threading.Thread(target=self._poll, args=(lib, h), daemon=True)
            self.thread.start()
            return self
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.source = "nvidia-smi, 20 ms"
        except (OSError, ValueError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        self._stop = True
        if self.thread is not None:
            self.thread.join(timeout=5)
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        if self.thread is not None:
            t0, t1 = self.window
            inside = [s for s in self.samples
                      if (t0 is None or s[0] >= t0) and (t1 is None or s[0] <= t1)]
            if not inside:
                return {"sm_mhz": None, "sm_max_mhz": self.sm_max, "reasons": ["no sample"],
                        "samples": 0, "source": self.source}
            names = sorted({nm for s in inside for bit, nm in self.REASONS.items() if s[3] & bit})
            pw = [s[2] for s in inside if s[2] is not None]
            return {"sm_mhz": statistics.median(s[1] for s in inside), "sm_max_mhz": self.sm_max,
                    "sm_mhz_min": min(s[1] for s in inside), "reasons": names,
                    "samples": len(inside), "power_w_max": max(pw) if pw else None,
                    "source": self.source}
        rows = [r for r in csv.reader(io.StringIO(self.out or "")) if len(r) >= 9]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        pw = [float(r[3]) for r in rows if r[3].strip().replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(pw) if pw else None, "source": self.source}


def dist_setup(n_gpus, backend=None):
    """Rank, world size and local rank from the torchrun environment; joins the
    process group when world > 1 (NCCL with a GPU per rank, gloo otherwise)."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if backend is None:
            backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """The maximum of x over all ranks (the slowest rank's time)."""
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job(units_per_rank: float, world: int, max_ms: float, steps: int):
    """Weak scaling: every rank processes units_per_rank per step; the job's rate
    is all ranks' units over the slowest rank's time (ms for `steps` steps)."""
    ms_per_step = max_ms / steps
    return world * units_per_rank / (ms_per_step * 1e-3), ms_per_step


# ------------------------------------------------------------------ the step
class Prefill:
    """Device-resident inputs/outputs of one projection's prefill step."""

    def __init__(self, tq, n, k, m, g, seed, act=torch.bfloat16, out=torch.float32):
        gen = torch.Generator(device="cuda")
        gen.manual_seed(seed)
        self.tq, self.n, self.k, self.m, self.g = tq, n, k, m, g
        self.w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
        self.x = torch.randn((m, k), generator=gen, device="cuda").to(act)
        self.dy = (torch.randn((m, n), generator=gen, device="cuda") * 1e-2).to(act)
        self.codes = torch.empty((n, k // 16), dtype=torch.int32, device="cuda")
        self.codes_t = torch.empty((k, 4 * ((n + 63) // 64)), dtype=torch.int32, device="cuda")
        self.s = torch.empty((n, k // g), dtype=torch.float32, device="cuda")
        self.z = torch.empty((n, k // g), dtype=torch.int32, device="cuda")
        self.y = torch.empty((m, n), dtype=out, device="cuda")
        self.dx = torch.empty((m, k), dtype=out, device="cuda")
        self.dw = torch.empty((n, k), dtype=torch.float32, device="cuda")

    @property
    def flops(self):
        return 3 * 2.0 * self.m * self.n * self.k

    def quantize_bytes(self):
        n, k, g = self.n, self.k, self.g
        return n * k * 4 + n * k // 4 + 2 * 4 * n * k // g

    def quantize_t_bytes(self):
        """The fused quantize's algorithmic bytes: those of quantize and the transposed
        codes written."""
        return self.quantize_bytes() + self.codes_t.numel() * 4

    def step(self, ev=None):
        tq = self.tq
        rec = (lambda i: ev[i].record()) if ev is not None else (lambda i: None)
        rec(0)
        tq.quantize_with_transpose(self.w, self.g, out=(self.codes, self.s, self.z, self.codes_t))
        rec(1)
        tq.linear_fwd(self.x, self.codes, self.s, self.g, y=self.y)
        rec(2)
        tq.linear_bwd(self.dy, self.x, self.codes, self.s, self.k, self.g, want_dw=False,
                      dx=self.dx, codes_t=self.codes_t)
        rec(3)
        tq.linear_bwd(self.dy, self.x, self.codes, self.s, self.k, self.g, want_dx=False,
                      dw=self.dw)
        rec(4)


KERNELS = [  # name, source files, event span
    ("quantize", ["quantize.cu", "ptx.cuh", "kernels.cuh", "quant_code.cuh"], (0, 1)),  # with the transpose
    ("fwd", ["ts_gemm.cu", "ptx.cuh", "kernels.cuh"], (1, 2)),
    ("dx", ["ts_gemm.cu", "ptx.cuh", "kernels.cuh"], (2, 3)),
    ("dw", ["dw_gemm.cu", "ptx.cuh", "kernels.cuh"], (3, 4)),
]


def time_prefill(p: Prefill, steps, warmup, world, clk=None):
    for _ in range(warmup):
        p.step()
    torch.cuda.synchronize()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(steps)]
    barrier(world)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    if clk is not None:
        clk.mark(True)
    t0.record()
    for i in range(steps):
        p.step(evs[i])
    t1.record()
    torch.cuda.synchronize()
    if clk is not None:
        clk.mark(False)
    barrier(world)
    total_ms = t0.elapsed_time(t1)
    per = {}
    for name, _, (a, b) in KERNELS:
        per[name] = sum(e[a].elapsed_time(e[b]) for e in evs) / steps
    p.tq.device_status()
    return total_ms, per


def roofline(per, total_ms, steps, pk, pk_kind, gemm_flops, quantize_bytes):
    """Per-kernel rates and the line's ``roofline`` object from the kernels' mean
    CUDA-event times ``per`` (ms) inside a timed region of ``total_ms`` over ``steps``.

    The measured peaks are a burst (best of 10 GEMMs) and a sustained figure (4 s of
    back-to-back GEMMs at the power cap): a timed region of under a second takes the
    burst peak, a longer one the sustained peak. The quantize is scored against HBM;
    the roofline reports the slowest GEMM, with the DRAM traffic of its committed ncu
    capture when its sources are unchanged."""
    region_s = total_ms / 1e3
    sustained = region_s >= 1.0
    tc_peak = pk["bf16_tflops_sustained"] if sustained else pk["bf16_tflops"]
    peak_rule = (f"{pk_kind} bf16 dense {'sustained' if sustained else 'burst'}: the timed region "
                 f"({steps} steps) lasted {region_s * 1e3:.1f} ms, "
                 f"{'at least' if sustained else 'under'} 1 s")
    kinfo = {}
    for name, files, _ in KERNELS:
        t = per[name]
        if name == "quantize":
            ach = quantize_bytes / (t * 1e-3) / 1e9
            kinfo[name] = {"ms": round(t, 4), "achieved": round(ach, 1), "unit": "GB/s",
                           "frac": round(ach / pk["hbm_gbs"], 4)}
        else:
            ach = gemm_flops / (t * 1e-3) / 1e12
            kinfo[name] = {"ms": round(t, 4), "achieved": round(ach, 1), "unit": "TFLOP/s",
                           "frac": round(ach / tc_peak, 4),
                           "frac_of_burst": round(ach / pk["bf16_tflops"], 4),
                           "frac_of_sustained": round(ach / pk["bf16_tflops_sustained"], 4)}
    dom = max((n for n, _, _ in KERNELS if n != "quantize"), key=lambda n: per[n])
    dom_files = dict((n, f) for n, f, _ in KERNELS)[dom]
    roof = {"kernel": dom, "bound": "tensor", "achieved": kinfo[dom]["achieved"],
            "peak": tc_peak, "unit": "TFLOP/s", "frac": kinfo[dom]["frac"],
            "traffic": recorded_traffic(dom, dom_files),
            "peak_kind": peak_rule, "timed_region_ms": round(total_ms, 3),
            "frac_of_burst": kinfo[dom]["frac_of_burst"], "burst_peak": pk["bf16_tflops"],
            "frac_of_sustained": kinfo[dom]["frac_of_sustained"],
            "sustained_peak": pk["bf16_tflops_sustained"],
            "algorithmic_per_launch": gemm_flops,
            "achieved_how": "algorithmic flops per launch / mean CUDA-event time of the "
                            "kernel's launch inside the timed steps"}
    return kinfo, roof


def time_e2e(p: Prefill, steps, warmup):
    """Same step through the C ABI from pinned host buffers: every step uploads its
    inputs (W, X, dY) and reads back all its outputs (Y, dX, dW) inside the timed
    region. As in a training loop, the copies of neighbouring steps overlap the
    compute: uploads on one stream, the step on a second, downloads on a third, over
    two device buffer sets ordered by events."""
    h_w = p.w.cpu().pin_memory()
    h_x = p.x.cpu().pin_memory()
    h_dy = p.dy.cpu().pin_memory()
    h_y = torch.empty(p.y.shape, dtype=p.y.dtype).pin_memory()
    h_dx = torch.empty(p.dx.shape, dtype=p.dx.dtype).pin_memory()
    h_dw = torch.empty(p.dw.shape, dtype=p.dw.dtype).pin_memory()
    q = Prefill.__new__(Prefill)
    q.__dict__.update({a: (v.clone() if torch.is_tensor(v) else v) for a, v in p.__dict__.items()})
    sets = (p, q)
    up, comp, down = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = {(name, j): torch.cuda.Event() for name in ("up", "comp", "down") for j in (0, 1)}

    def issue(i):
        j = i % 2
        b = sets[j]
        with torch.cuda.stream(up):
            if i >= 2:
                up.wait_event(ev["comp", j])  # set j's inputs are free
            b.w.copy_(h_w, non_blocking=True)
            b.x.copy_(h_x, non_blocking=True)
            b.dy.copy_(h_dy, non_blocking=True)
            ev["up", j].record(up)
        with torch.cuda.stream(comp):
            comp.wait_event(ev["up", j])
            if i >= 2:
                comp.wait_event(ev["down", j])  # set j's outputs were read back
            b.step()
            ev["comp", j].record(comp)
        with torch.cuda.stream(down):
            down.wait_event(ev["comp", j])
            h_y.copy_(b.y, non_blocking=True)
            h_dx.copy_(b.dx, non_blocking=True)
            h_dw.copy_(b.dw, non_blocking=True)
            ev["down", j].record(down)

    for i in range(warmup):
        issue(i)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(up)
    for i in range(steps):
        issue(i)
    t1.record(down)  # the last download waits for every earlier operation
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / steps
    h2d = sum(t.numel() * t.element_size() for t in (h_w, h_x, h_dy))
    d2h = sum(t.numel() * t.element_size() for t in (h_y, h_dx, h_dw))
    return ms, h2d, d2h


def _decode_mats(tq, gen):
    """The packed in_proj and out_proj of all 48 layers, layer by layer."""
    mats = []
    for layer in range(N_LAYERS):
        for (n, k) in (IN_PROJ, OUT_PROJ):
            w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
            codes, s, _ = tq.quantize(w, G)
            mats.append((n, k, codes, s))
            del w
    return mats


def decode_sweep(tq, m_list, steps, warmup):
    """Decode forward over all 48 layers' packed in_proj and out_proj (one batched call)."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(1234)
    mats = _decode_mats(tq, gen)
    out = {}
    for m in m_list:
        items = []
        for (n, k, codes, s) in mats:
            x = torch.randn((m, k), generator=gen, device="cuda").to(torch.bfloat16)
            items.append(dict(x=x, codes=codes, scales=s, g=G,
                              y=torch.empty((m, n), device="cuda")))
        arr = tq.fwd_batch(items)  # descriptors built once, outside the timed loop
        for _ in range(warmup):
            tq.linear_fwd_batched(arr, m)
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(steps):
            tq.linear_fwd_batched(arr, m)
        t1.record()
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / steps
        nbytes = sum(it["codes"].numel() * 4 + it["scales"].numel() * 4 + it["x"].numel() * 2 +
                     it["y"].numel() * 4 for it in items)
        out[f"M={m}"] = {"us": round(ms * 1e3, 2), "GB/s": round(nbytes / ms / 1e6, 1),
                         "bytes": nbytes}
    tq.device_status()
    return out


def decode_per_layer(tq, m_list, replays, warmup):
    """One decode step as a model runs it: layer after layer, in_proj then out_proj,
    one tq_linear_fwd launch each (96 launches in stream order), captured once in a
    CUDA graph and replayed, so that the host's per-call cost stays out of the
    device time. The 351 MB of codes exceed L2: every replay streams them from HBM."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(4321)
    mats = _decode_mats(tq, gen)
    out = {}
    for m in m_list:
        calls = []
        for (n, k, codes, s) in mats:
            x = torch.randn((m, k), generator=gen, device="cuda").to(torch.bfloat16)
            calls.append((x, codes, s, torch.empty((m, n), device="cuda")))
        stream = torch.cuda.Stream()
        stream.wait_stream(torch.cuda.current_stream())

        def step():
            for (x, codes, s, y) in calls:
                tq.linear_fwd(x, codes, s, G, y=y, stream=stream)

        with torch.cuda.stream(stream):
            step()  # outside the capture: attributes, tensor maps, cluster sizes
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            step()
        for _ in range(warmup):
            graph.replay()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(replays):
            graph.replay()
        t1.record()
        torch.cuda.synchronize()
        us = t0.elapsed_time(t1) * 1e3 / replays
        nbytes = sum(c.numel() * 4 + s_.numel() * 4 + x.numel() * 2 + y.numel() * 4
                     for (x, c, s_, y) in calls)
        out[f"M={m}"] = {"us_per_step": round(us, 1), "us_per_layer": round(us / N_LAYERS, 2),
                         "launches": len(calls), "GB/s": round(nbytes / us / 1e3, 1)}
        del graph
    tq.device_status()
    return out


def quantize_sweep(tq, steps, warmup):
    """tq_quantize_batched over the 96 projections of 48 blocks in one launch (the
    per-step requantize)."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(99)
    ws = [torch.randn(shape, generator=gen, device="cuda") * 0.02
          for _ in range(N_LAYERS) for shape in (IN_PROJ, OUT_PROJ)]
    outs = [(torch.empty((w.shape[0], w.shape[1] // 16), dtype=torch.int32, device="cuda"),
             torch.empty((w.shape[0], w.shape[1] // G), device="cuda"),
             torch.empty((w.shape[0], w.shape[1] // G), dtype=torch.int32, device="cuda"))
            for w in ws]

    arr = tq.quant_batch([(w, *o) for w, o in zip(ws, outs)])

    def run():
        tq.quantize_batched(arr, G)

    for _ in range(warmup):
        run()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(steps):
        run()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / steps
    nbytes = sum(w.numel() * 4 + w.numel() // 4 + 2 * 4 * w.numel() // G for w in ws)
    tq.device_status()
    del ws, outs
    return {"ms": round(ms, 3), "GB/s": round(nbytes / ms / 1e6, 1), "bytes": nbytes}


def out_proj_step(tq, steps, warmup, shape=OUT_PROJ, act=torch.bfloat16, out=torch.float32):
    """The same step on another shape (default out_proj: W [2048, 4096], X [16384, 4096]),
    activation type or output type of Y and dX."""
    p = Prefill(tq, shape[0], shape[1], M_PREFILL, G, seed=8, act=act, out=out)
    total_ms, per = time_prefill(p, steps, warmup, 1)
    ms = total_ms / steps
    gemm = 2.0 * p.m * p.n * p.k
    out = {"ms": round(ms, 4), "TFLOP/s": round(p.flops / ms / 1e9, 1)}
    for name in ("fwd", "dx", "dw"):
        out[name] = {"ms": round(per[name], 4), "TFLOP/s": round(gemm / per[name] / 1e9, 1)}
    out["quantize"] = {"ms": round(per["quantize"], 4),
                       "GB/s": round(p.quantize_t_bytes() / per["quantize"] / 1e6, 1)}
    del p
    return out


def student_t3(shape, gen, std):
    """Student-t with 3 degrees of freedom scaled to standard deviation std: z / sqrt(chi2_3 / 3),
    the variance of t_3 being 3."""
    z = torch.randn(shape, generator=gen, device="cuda")
    c = sum(torch.randn(shape, generator=gen, device="cuda") ** 2 for _ in range(3)) / 3.0
    return z / c.sqrt() * (std / math.sqrt(3.0))


def g_sweep(tq):
    """The 48-block sweep at batch 8 x seq 2048 for every group size and both weight
    distributions: per (distribution, g) one batched requantize of the 96 projections,
    then per projection the codes transpose, forward, dX and dW. X and dY are shared by
    the layers of a projection type (the GEMMs are compute-bound)."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    shapes = [IN_PROJ, OUT_PROJ] * N_LAYERS
    act = {}
    for n, k in (IN_PROJ, OUT_PROJ):
        act[(n, k)] = dict(
            x=torch.randn((M_PREFILL, k), generator=gen, device="cuda").to(torch.bfloat16),
            dy=(torch.randn((M_PREFILL, n), generator=gen, device="cuda") * 1e-2).to(torch.bfloat16),
            y=torch.empty((M_PREFILL, n), device="cuda"),
            dx=torch.empty((M_PREFILL, k), device="cuda"),
            dw=torch.empty((n, k), device="cuda"))
    flops = sum(3 * 2.0 * M_PREFILL * n * k for n, k in shapes)
    pk, _ = peaks()
    res = {}
    for dist in ("gauss", "t3"):
        ws = [(torch.randn(sh, generator=gen, device="cuda") * 0.02) if dist == "gauss"
              else student_t3(sh, gen, 0.02) for sh in shapes]
        codes = [torch.empty((n, k // 16), dtype=torch.int32, device="cuda") for n, k in shapes]
        codes_t = [torch.empty((k, 4 * ((n + 63) // 64)), dtype=torch.int32, device="cuda")
                   for n, k in shapes]
        for g in (32, 64, 128, 256, 512):
            sc = [torch.empty((n, k // g), device="cuda") for n, k in shapes]
            zs = [torch.empty((n, k // g), dtype=torch.int32, device="cuda") for n, k in shapes]
            arr = tq.quant_batch([(w, c, s_, z) for w, c, s_, z in zip(ws, codes, sc, zs)])

            def gemms():
                for (n, k), c, ct, s_ in zip(shapes, codes, codes_t, sc):
                    a = act[(n, k)]
                    tq.codes_transpose(c, k, out=ct)
                    tq.linear_fwd(a["x"], c, s_, g, y=a["y"])
                    tq.linear_bwd(a["dy"], a["x"], c, s_, k, g, want_dw=False, dx=a["dx"], codes_t=ct)
                    tq.linear_bwd(a["dy"], a["x"], c, s_, k, g, want_dx=False, dw=a["dw"])

            tq.quantize_batched(arr, g)
            gemms()
            torch.cuda.synchronize()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            ev[0].record()
            tq.quantize_batched(arr, g)
            ev[1].record()
            gemms()
            ev[2].record()
            torch.cuda.synchronize()
            tq.device_status()
            q_ms, g_ms = ev[0].elapsed_time(ev[1]), ev[1].elapsed_time(ev[2])
            numel = sum(n * k for n, k in shapes)
            qbytes = numel * 4 + numel // 4 + 2 * 4 * numel // g
            zero = sum(int(z.sum(dtype=torch.int64)) for z in zs) / numel
            ach = flops / g_ms / 1e9
            res[f"{dist}_g{g}"] = {
                "quantize_ms": round(q_ms, 3), "quantize_GB/s": round(qbytes / q_ms / 1e6, 1),
                "quantize_frac": round(qbytes / q_ms / 1e6 / pk["hbm_gbs"], 4),
                "gemms_ms": round(g_ms, 2), "TFLOP/s": round(ach, 1),
                "frac": round(ach / pk["bf16_tflops"], 4), "zero_ratio": round(zero, 4)}
            del sc, zs, arr
        del ws, codes, codes_t
    res["note"] = ("per (distribution, g): one batched requantize of the 96 projections, then "
                   "codes transpose + forward + dX + dW of every projection; "
                   f"{flops / 1e12:.2f} TFLOP of GEMMs per sweep")
    return res


def adamw_sweep(tq, steps, warmup):
    """tq_adamw_requantize (AdamW step + requantize, g = 128) on the in_proj matrix
    alone and over the 96 projections of the 48 blocks (one launch each): per weight
    16 B read (w, grad, m, v) and 12 B + codes + scale and count written."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(31)
    pk, _ = peaks()
    hp = dict(lr=2.5e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01)

    def state(n, k):
        w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
        g = torch.randn((n, k), generator=gen, device="cuda") * 1e-3
        m = torch.zeros((n, k), device="cuda")
        v = torch.zeros((n, k), device="cuda")
        out = (torch.empty((n, k // 16), dtype=torch.int32, device="cuda"),
               torch.empty((n, k // G), device="cuda"),
               torch.empty((n, k // G), dtype=torch.int32, device="cuda"))
        return w, g, m, v, out

    def per_weight_bytes():
        return 28 + 0.25 + 8.0 / G

    res = {}
    for label, shapes in (("in_proj", [IN_PROJ]), ("48_layers", [IN_PROJ, OUT_PROJ] * N_LAYERS)):
        mats = [state(n, k) for n, k in shapes]
        t = [0]

        def run():
            t[0] += 1
            for w, g, m, v, out in mats:
                tq.adamw_requantize(w, g, m, v, G, step=t[0], out=out, **hp)

        for _ in range(warmup):
            run()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(steps):
            run()
        t1.record()
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / steps
        nbytes = sum(n * k for n, k in shapes) * per_weight_bytes()
        res[label] = {"ms": round(ms, 4), "GB/s": round(nbytes / ms / 1e6, 1),
                      "frac": round(nbytes / ms / 1e6 / pk["hbm_gbs"], 4), "bytes": int(nbytes)}
        del mats
    tq.device_status()
    return res


def decoupled_sweep(tq, steps, warmup):
    """The decoupled quantizer on in_proj with the asymmetric gate (rows 0..4095 at
    0.8 x absmean), and the magnitude gradient dalpha = sum dW * c per group."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(41)
    pk, _ = peaks()
    n, k = IN_PROJ
    w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
    dw = torch.randn((n, k), generator=gen, device="cuda")
    f = torch.ones(n, device="cuda")
    f[:4096] = 0.8
    out = (torch.empty((n, k // 16), dtype=torch.int32, device="cuda"),
           torch.empty((n, k // G), device="cuda"),
           torch.empty((n, k // G), dtype=torch.int32, device="cuda"))
    da = torch.empty((n, k // G), device="cuda")
    res = {}
    for label, fn, nbytes in (
            ("quantize_decoupled", lambda: tq.quantize_decoupled(w, G, f, out=out),
             n * k * 4 + n * k // 4 + 8 * n * k // G + 4 * n),
            ("alpha_grad", lambda: tq.alpha_grad(dw, out[0], G, out=da),
             n * k * 4 + n * k // 4 + 4 * n * k // G)):
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(steps):
            fn()
        t1.record()
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / steps
        res[label] = {"us": round(ms * 1e3, 2), "GB/s": round(nbytes / ms / 1e6, 1),
                      "frac": round(nbytes / ms / 1e6 / pk["hbm_gbs"], 4), "bytes": nbytes}
    zr = out[2].double()
    res["zero_ratio_gate_rows"] = round(float(zr[:4096].mean()) / G, 4)
    res["zero_ratio_other_rows"] = round(float(zr[4096:].mean()) / G, 4)
    tq.device_status()
    return res


def learnable_sweep(tq, steps, warmup):
    """The learnable-scale variant on in_proj: codes against given scales, the
    scale gradient, and the fused AdamW step with requantization against given
    scales; then the zero ratio of both scale parameterizations over a synthetic
    teacher-student run (paper_2606_18114_gb300.qat) on the out_proj shape."""
    from paper_2606_18114_gb300 import qat
    gen = torch.Generator(device="cuda")
    gen.manual_seed(43)
    pk, _ = peaks()
    n, k = IN_PROJ
    w = torch.randn((n, k), generator=gen, device="cuda") * 0.02
    dw = torch.randn((n, k), generator=gen, device="cuda") * 1e-3
    m, v = torch.zeros_like(w), torch.randn((n, k), generator=gen, device="cuda").abs() * 1e-7
    codes, s, z = tq.quantize(w, G)
    s.mul_(1.1)
    ds = torch.empty_like(s)
    res = {}
    for label, fn, nbytes in (
            ("quantize_with_scales", lambda: tq.quantize_with_scales(w, G, s, out=(codes, z)),
             n * k * 4 + n * k // 4 + 8 * n * k // G),
            ("scale_grad", lambda: tq.scale_grad(w, dw, codes, s, G, out=ds),
             2 * n * k * 4 + n * k // 4 + 8 * n * k // G),
            ("adamw_requantize_with_scales",
             lambda: tq.adamw_requantize_with_scales(w, dw, m, v, G, s, lr=1e-9, step=1,
                                                     out=(codes, z)),
             28 * n * k + n * k // 4 + 8 * n * k // G)):
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(steps):
            fn()
        t1.record()
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / steps
        res[label] = {"us": round(ms * 1e3, 2), "GB/s": round(nbytes / ms / 1e6, 1),
                      "frac": round(nbytes / ms / 1e6 / pk["hbm_gbs"], 4), "bytes": nbytes}
    tq.device_status()
    on, ok = OUT_PROJ
    steps = 2000
    track = {}
    for lr in (2.5e-4, 5e-5, 1e-5):
        per = {}
        for label, learnable in (("fixed_absmean", False), ("learnable_scale", True)):
            rows = qat.track_zero_ratio(tq, on, ok, 1024, G, steps, learnable, seed=5, lr=lr,
                                        every=400)
            per[label] = [{kk: (round(vv, 7) if kk == "loss" else vv) for kk, vv in r.items()}
                          for r in rows]
        track[f"lr_{lr:g}"] = per
    res["zero_ratio_tracking"] = {
        "task": f"teacher-student regression, W [{on}, {ok}] g={G}, 1024 tokens per step, "
                f"{steps} AdamW steps (beta 0.9/0.95, decay 0.01) at each peak lr, linear "
                f"warm-up over {steps // 50} steps then cosine decay to 0, student from the "
                "teacher's weights",
        **track}
    return res


def cublas_context(tq):
    """cuBLAS bf16 dense GEMM of the forward's shape (Y = X W^T, 16384 x 8512 x 2048):
    context for the tensor-core fraction, not part of the path."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(3)
    x = torch.randn((M_PREFILL, IN_PROJ[1]), generator=gen, device="cuda").to(torch.bfloat16)
    w = torch.randn(IN_PROJ, generator=gen, device="cuda").to(torch.bfloat16)
    for _ in range(3):
        torch.matmul(x, w.t())
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(20):
        torch.matmul(x, w.t())
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / 20
    return {"ms": round(ms, 4),
            "TFLOP/s": round(2.0 * M_PREFILL * IN_PROJ[0] * IN_PROJ[1] / ms / 1e9, 1),
            "note": "torch.matmul bf16 (cuBLAS), bf16 output; context only"}


# ------------------------------------------------------------------ oracle (CPU)
def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return len(os.sched_getaffinity(0))


def oracle_sample(seed=0):
    """A bounded sample of one step, run by the oracle on the host cores.

    Quantises the full W [8512, 2048] and computes Y and dX for 64 token rows and
    dW for 64 output rows (fp64). Returns (flops of the sample, seconds).
    """
    from oracle import tq_oracle as O
    from paper_2606_18114_gb300 import synth
    n, k = IN_PROJ
    w = synth.latent_weights(n, k, seed=seed)
    rs = np.random.default_rng(seed)
    rows = 64
    x = synth.activations_bf16(M_PREFILL, k, seed=seed, stream="x")
    dy_rows = synth.activations_bf16(rows, n, seed=seed, std=1e-2, stream="dy_sample")
    nsel = np.sort(rs.choice(n, rows, replace=False))
    dy_cols = synth.activations_bf16(M_PREFILL, rows, seed=seed, std=1e-2, stream="dy_cols")
    t0 = time.perf_counter()
    codes, s, z, _ = O.quantize(w, G)
    w_hat = O.dequantize(codes, s, k, G)
    O.linear_fwd(x[:rows], w_hat)
    O.linear_bwd_dx(dy_rows, w_hat)
    O.linear_bwd_dw(dy_cols, x)
    dt = time.perf_counter() - t0
    flops = 2.0 * rows * n * k * 2 + 2.0 * rows * M_PREFILL * k
    del nsel
    return flops, dt


def cpu_baseline():
    flops, dt = oracle_sample()
    return {"value": round(flops / dt / 1e12, 6), "unit": "TFLOP/s", "cores": blas_threads(),
            "kind": "oracle",
            "sample": ("oracle (numpy, fp64) on one step's bounded sample: quantize the full "
                       "W[8512,2048] g=128, then Y and dX for 64 of 16384 token rows and dW for "
                       "64 of 8512 output rows; flops of the sample / wall time"),
            "seconds": round(dt, 2)}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    for _ in range(args.warmup):
        oracle_sample()
    times, flops = [], 0.0
    for _ in range(args.steps):
        f, dt = oracle_sample()
        flops, times = f, times + [dt]
    dt = sum(times) / len(times)
    value = flops / dt / 1e12
    line = {
        "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s", "impl": "reference",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt * 1e3, 1), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "M": M_PREFILL, "N": IN_PROJ[0], "K": IN_PROJ[1],
                   "g": G, "sample": "bounded oracle sample per step (see cpu_baseline)"},
        "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": blas_threads(),
                         "kind": "oracle",
                         "sample": "quantize full W; Y, dX on 64 token rows; dW on 64 output rows"},
        "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_only(args):
    """One kernel of the step in isolation (for ncu captures of a single launch)."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_18114_gb300 import tq
    torch.cuda.set_device(0)
    if args.only == "decode":
        res = decode_sweep(tq, (1,), args.steps, args.warmup)
        print(json.dumps({"only": "decode", **res}), flush=True)
        return
    if args.only == "decode_single":
        # one in_proj projection at one token, one launch per call (k cut into pieces)
        n, k = IN_PROJ
        w = torch.randn((n, k), device="cuda") * 0.02
        codes, s, _ = tq.quantize(w, G)
        x = torch.randn((1, k), device="cuda").to(torch.bfloat16)
        y = torch.empty((1, n), device="cuda")
        for _ in range(args.warmup + args.steps):
            tq.linear_fwd(x, codes, s, G, y=y)
        torch.cuda.synchronize()
        tq.device_status()
        print(json.dumps({"only": "decode_single", "n": n, "k": k, "m": 1}), flush=True)
        return
    if args.only == "adamw":
        n, k = IN_PROJ
        w = torch.randn((n, k), device="cuda") * 0.02
        gr = torch.randn((n, k), device="cuda") * 1e-3
        m = torch.zeros((n, k), device="cuda")
        v = torch.zeros((n, k), device="cuda")
        step = [0]

        def upd():
            step[0] += 1
            tq.adamw_requantize(w, gr, m, v, G, lr=2.5e-4, step=step[0])
        calls = {"adamw": upd}
    else:
        calls = {}
    p = Prefill(tq, IN_PROJ[0], IN_PROJ[1], M_PREFILL, G, seed=7)
    tq.quantize(p.w, p.g, out=(p.codes, p.s, p.z))
    tq.codes_transpose(p.codes, p.k, out=p.codes_t)
    dwr = torch.randn((p.n, p.k), device="cuda") * 1e-3
    sg = p.s * 1.1  # given scales of the learnable-scale variant
    ds, da = torch.empty_like(p.s), torch.empty_like(p.s)
    calls.update({
        "given": lambda: tq.quantize_with_scales(p.w, p.g, sg, out=(p.codes, p.z)),
        "scale_grad": lambda: tq.scale_grad(p.w, dwr, p.codes, sg, p.g, out=ds),
        "alpha_grad": lambda: tq.alpha_grad(dwr, p.codes, p.g, out=da),
        "quantize": lambda: tq.quantize(p.w, p.g, out=(p.codes, p.s, p.z)),
        "quantize_t": lambda: tq.quantize_with_transpose(p.w, p.g,
                                                         out=(p.codes, p.s, p.z, p.codes_t)),
        "transpose": lambda: tq.codes_transpose(p.codes, p.k, out=p.codes_t),
        "fwd": lambda: tq.linear_fwd(p.x, p.codes, p.s, p.g, y=p.y),
        "dx": lambda: tq.linear_bwd(p.dy, p.x, p.codes, p.s, p.k, p.g, want_dw=False, dx=p.dx,
                                    codes_t=p.codes_t),
        "dw": lambda: tq.linear_bwd(p.dy, p.x, p.codes, p.s, p.k, p.g, want_dx=False, dw=p.dw),
    })
    fn = calls[args.only]
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        fn()
    t1.record()
    torch.cuda.synchronize()
    tq.device_status()
    print(json.dumps({"only": args.only, "ms": t0.elapsed_time(t1) / max(args.steps, 1)}),
          flush=True)


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="tq", choices=["tq", "reference"])
    ap.add_argument("--no-extra", action="store_true", help="skip decode/quantize sweeps")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--only", choices=["quantize", "quantize_t", "transpose", "fwd", "dx", "dw", "decode",
                                       "decode_single", "adamw",
                                       "given", "scale_grad", "alpha_grad"],
                    help="profiling aid: run just this kernel of the step (or the batched "
                         "M=1 decode) --warmup + --steps times and print its time")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.only:
        run_only(args)
        return
    if args.warmup < 3:
        args.warmup = 3

    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_18114_gb300 import tq

    rank, world, local = dist_setup(args.gpus)
    p = Prefill(tq, IN_PROJ[0], IN_PROJ[1], M_PREFILL, G, seed=1000 + rank)
    with ClockSampler(local) as clk:
        total_ms, per = time_prefill(p, args.steps, args.warmup, world, clk)
    total_ms = max_over_ranks(total_ms, world)
    rate, ms = whole_job(p.flops, world, total_ms, args.steps)
    value = rate / 1e12

    pk, pk_kind = peaks()
    kinfo, roof = roofline(per, total_ms, args.steps, pk, pk_kind, 2.0 * p.m * p.n * p.k,
                           p.quantize_t_bytes())

    # enough steps that filling and draining the copy pipeline (the first upload and
    # compute, the last download) stay a small share of the timed region
    e2e_steps = max(10, args.steps // 2)
    barrier(world)
    e2e_ms, h2d, d2h = time_e2e(p, e2e_steps, 2)
    barrier(world)
    e2e_rate, e2e_ms = whole_job(p.flops, world, max_over_ranks(e2e_ms * e2e_steps, world),
                                 e2e_steps)
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "M": M_PREFILL, "N": IN_PROJ[0], "K": IN_PROJ[1],
                   "g": G, "w_dist": "N(0,0.02^2)", "x_dist": "N(0,1) bf16",
                   "dy_dist": "N(0,1e-2^2) bf16", "outputs": "Y, dX fp32; dW fp32",
                   "l2": "no flush: every step reads and writes > 1 GB (inputs exceed the 129 MB L2)",
                   "replicas": world},
        "roofline": roof,
        "kernels": kinfo,
        "e2e": {"value": round(e2e_rate / 1e12, 2), "unit": "TFLOP/s",
                "ms_per_step": round(e2e_ms, 3), "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                "overlap": "uploads, step and downloads of neighbouring steps on three streams",
                "note": ("bound by the host link: every step reads back Y (fp32, 558 MB), dX (fp32, "
                         "134 MB) and dW (fp32, 70 MB); the outputs stay fp32 so that the maximum "
                         "element error against the oracle stays small")},
        "gpu_launches": len(KERNELS) * args.steps,
        "clocks": clk.summary(),
    }
    if not args.no_extra and rank == 0:
        line["extra"] = {
            "decode_48_layers": decode_sweep(tq, (1, 4, 16), 20, 3),
            "decode_48_layers_launch_per_projection": decode_per_layer(tq, (1, 4, 16), 20, 3),
            "quantize_48_layers_g128": quantize_sweep(tq, 5, 2),
            "out_proj_step": out_proj_step(tq, 200, 10),
            "in_proj_step_fp16_activations": out_proj_step(tq, 200, 10, IN_PROJ, torch.float16),
            "in_proj_step_bf16_outputs": out_proj_step(tq, 200, 10, IN_PROJ, out=torch.bfloat16),
            "sweep_48_layers": g_sweep(tq),
            "adamw_requantize_g128": adamw_sweep(tq, 5, 2),
            "decoupled_in_proj": decoupled_sweep(tq, 20, 3),
            "learnable_scale_in_proj": learnable_sweep(tq, 20, 3),
            "cublas_bf16_fwd_shape": cublas_context(tq),
            "hbm_peak_gbs": pk["hbm_gbs"],
        }
    if rank == 0 and world == 1 and not args.no_cpu:
        line["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
