#!/usr/bin/env python
"""Throughput of the quaternion convolution forward (libquan) on synthetic layers.

One step = one full pass of the hot path (staging, on-chip Hamilton block expansion,
contraction, bias/IQBN/activation epilogue, store) over one batch of the workload.
Default workload: the ResNet-18-style QUAN backbone forward, N=256 images of 224x224x4
quaternion input, 20 quaternion convolutions with fused IQBN + ReLU and the stem's 3x3/2
max pool, bf16 in / fp32 accumulate, in images/s (--act silu, --no-fuse).  Other
workloads: --workload c1 (the CIFAR-shaped layer N=128, 32x32, 64->64 real channels,
3x3 s1 p1) | c2a | c2b | c3a | c3b (ImageNet / detection-neck layers), in real-equivalent
TFLOP/s | poincare (the Eq. 4 input mapping) | iqbn (training-mode IQBN); on a layer
workload, --variant separable (Eq. 7) and --pass bwd (the input and weight gradients).

Prints one JSON line.  Under torchrun every rank runs its own copy of the workload on
its own GPU (the batch shards with no exchange step: weak scaling); the timed region
is bracketed by a barrier and a device synchronisation and the max over ranks is taken.
--impl reference times the fp64 CPU oracle on the host cores instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "QConv fwd real-equiv TFLOP/s & % bf16 tensor peak (1 GB300); backbone images/s"
L2_BYTES = 126 * 1024 * 1024
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.070e9 / 1e12  # FFMA: SMs x lanes x 2 FLOP x max clock


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="backbone",
                    choices=["c1", "c2a", "c2b", "c3a", "c3b", "backbone", "poincare", "iqbn"])
    ap.add_argument("--pass", dest="direction", choices=["fwd", "bwd"], default="fwd",
                    help="layer workloads: the forward convolution, or its backward pass "
                         "(input and weight gradients before the epilogue, from a seeded "
                         "output gradient)")
    ap.add_argument("--variant", choices=["full", "separable"], default="full",
                    help="layer workloads: the full Hamilton form (Eq. 5/6) or the separable "
                         "form of Eq. 7 (a quarter of the multiply-adds)")
    ap.add_argument("--act", choices=["relu", "silu"], default="relu",
                    help="backbone: the activation of its convolutions (ReLU as configured, "
                         "or SiLU as in YOLO-style detectors)")
    ap.add_argument("--no-fuse", action="store_true",
                    help="backbone: run the stem and its max pool as two calls")
    ap.add_argument("--rgb", action="store_true",
                    help="backbone: start from fp32 RGB pixels, mapped to quaternions by Eq. 4 "
                         "inside the fused stem kernel's loader")
    ap.add_argument("--no-split", action="store_true",
                    help="backbone: run the convolutions without the split-K workspace "
                         "(quan_qconv2d_fwd / _res instead of quan_qconv2d_fwd_ex)")
    ap.add_argument("--no-overlap", action="store_true",
                    help="backbone: run every layer on one stream (by default each 1x1/2 "
                         "shortcut runs on a second stream beside the block's 3x3/2 "
                         "convolution, forked and joined by events)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=24.0,
                    help="target of the bounded oracle sample, sized from a one-image run "
                         "(the oracle's threads scale better on many images, so the sample "
                         "itself takes about half of it: ~10-12 s)")
    ap.add_argument("--profile", action="store_true",
                    help="for ncu: exactly W + K plain launches, no clock sampling, no e2e "
                         "or CPU legs")
    ap.add_argument("--no-graph", action="store_true",
                    help="time a plain launch loop instead of one CUDA-graph replay")
    ap.add_argument("--batch", type=int, default=0,
                    help="with --profile: run the workload at this batch size (a smaller "
                         "case for multi-pass ncu captures)")
    return ap.parse_args()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, \
            "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# host-side front end (argument checks, path choice): no device code, so editing it does
# not change what an ncu capture of a kernel measured
HOST_ONLY_SOURCES = ("quan_api.cu",)


# Device-code sources each kernel is built from, beyond the shared ones: an ncu traffic
# figure stays valid while these are unchanged.  qconv_tc.cu holds the tensor-core kernels'
# host launch code (grid, tiles, tensor maps) and includes every .cuh listed here.
SHARED_DEVICE_SOURCES = ("ptx.cuh", "tc_common.cuh", "internal.h")
KERNEL_SOURCES = {
    "qconv_stem_pool_kernel": ("qconv_tc.cu", "qconv_stempool.cuh", "qconv_gather.cuh"),
    "qconv_pairs_kernel": ("qconv_tc.cu", "qconv_gather.cuh"),
    "qconv_vs_kernel": ("qconv_tc.cu", "qconv_vs.cuh"),
    "qconv_ws_kernel": ("qconv_tc.cu", "qconv_ws.cuh"),
    "qconv_cg2_kernel": ("qconv_tc.cu", "qconv_cg2.cuh"),
    "qconv_pw_kernel": ("qconv_tc.cu", "qconv_pw.cuh"),
    "qconv_tc_kernel": ("qconv_tc.cu",),
    "qconv_dw_kernel": ("qconv_tc.cu", "qconv_dw.cuh"),
    "iqbn_apply_kernel": ("iqbn.cu",),
    "iqbn_stats_kernel": ("iqbn.cu",),
    "poincare_kernel": ("poincare.cu",),
}


def kernel_source_hash(kernel: str | None = None) -> str:
    """Hash of the device-code sources of `kernel` (the library's kernel name; its base
    name before '<' selects the files), or of every source under csrc but the host-only
    front end for an unknown or absent name."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2509_05512_gb300", "csrc")
    base = (kernel or "").split("<")[0].split()[0] if kernel else ""
    if base in KERNEL_SOURCES:
        names = sorted(SHARED_DEVICE_SOURCES + KERNEL_SOURCES[base])
    else:
        names = [n for n in sorted(os.listdir(csrc)) if n not in HOST_ONLY_SOURCES]
    for name in names:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode())
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str, kernel: str | None = None, path: str | None = None):
    """DRAM bytes per launch of the dominant kernel from the committed ncu summary, or
    None when no capture exists, it is of another kernel or template instance (the full
    name, template arguments included, must match), or that kernel's device sources
    changed since it was taken."""
    path = path or os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(workload)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("kernel_sha") != kernel_source_hash(rec.get("kernel")):
        return None
    if kernel is not None and kernel != rec.get("kernel"):
        return None  # another kernel, or another template instance of it
    return rec.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling while the GPU is busy."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.proc = None
        self.file = tempfile.NamedTemporaryFile(mode="w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", gpu_id, "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [ln.strip().split(", ") for ln in self.file if ln.strip()]
        os.unlink(self.file.name)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
            except ValueError:
                continue
            for name, v in zip(names, r[5:9]):
                if v.strip() == "Active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------- layers

E2E_BUFFERS = 2  # device buffer sets of the end-to-end pipeline


def e2e_pipeline(runner, torch, stream, steps):
    """`steps` end-to-end steps through the public call.  Step k copies its inputs from
    pinned host memory (copy stream), runs the path on buffer set k % E2E_BUFFERS (compute
    stream) and copies its result back (second copy stream).  Events order every buffer
    set's uses, so step k's copies overlap the kernels of its neighbours; every step still
    moves all of its own bytes.  Returns once everything is queued; both copy streams join
    `stream` at the end, so events on `stream` bracket the whole run."""
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    s_in.wait_stream(stream)
    s_out.wait_stream(stream)
    nb = E2E_BUFFERS
    ev = lambda: [torch.cuda.Event() for _ in range(nb)]
    ev_in, ev_comp, ev_out = ev(), ev(), ev()
    sh = stream.cuda_stream
    for k in range(steps):
        b = k % nb
        if k >= nb:
            s_in.wait_event(ev_comp[b])  # step k - nb has consumed buffer set b's inputs
        with torch.cuda.stream(s_in):
            for dst, src in runner.e2e_in(b):
                dst.copy_(src, non_blocking=True)
        ev_in[b].record(s_in)
        stream.wait_event(ev_in[b])
        if k >= nb:
            stream.wait_event(ev_out[b])  # step k - nb's result has left buffer set b
        runner.e2e_compute(b, sh)
        ev_comp[b].record(stream)
        s_out.wait_event(ev_comp[b])
        with torch.cuda.stream(s_out):
            for dst, src in runner.e2e_out(b):
                dst.copy_(src, non_blocking=True)
        ev_out[b].record(s_out)
    stream.wait_stream(s_in)
    stream.wait_stream(s_out)


class LayerRunner:
    """Device buffers for one layer, rotated so that consecutive steps never find their
    inputs in L2."""

    def __init__(self, spec, torch, quan, inputs, separable=False):
        import numpy as np
        self.spec, self.torch, self.quan = spec, torch, quan
        self.separable = separable
        self.conv = quan.quan_qconv2d_sep_fwd if separable else quan.quan_qconv2d_fwd
        d = inputs.layer_inputs(spec)
        dev = torch.device("cuda")

        def up(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(
                torch.bfloat16).to(dev)

        self.host = d
        x0 = up(d["x"])
        self.w = [up(d[k]) for k in ("wr", "wi", "wj", "wk")]
        f32 = lambda a: None if a is None else torch.from_numpy(a).to(dev)
        self.bias, self.scale, self.shift = f32(d["bias"]), f32(d["scale"]), f32(d["shift"])
        out_elems = spec.N * spec.Ho * spec.Wo * spec.Cout
        per_set = (x0.numel() + out_elems) * 2
        self.sets = max(2, min(16, math.ceil(2 * L2_BYTES / per_set)))
        self.xs = [x0] + [x0.clone() for _ in range(self.sets - 1)]
        self.outs = [torch.empty((spec.N, spec.Ho, spec.Wo, spec.Cout), dtype=torch.bfloat16,
                                 device=dev) for _ in range(self.sets)]
        self.i = 0
        self.launches_per_step = 1
        self.footprint = per_set * self.sets

    def step(self, stream):
        s = self.spec
        k = self.i % self.sets
        self.i += 1
        self.conv(self.xs[k], *self.w, self.bias, self.scale, self.shift, s.N, s.H, s.W, s.Cin,
                  s.Cout, s.kh, s.kw, s.stride, s.pad, s.act, self.outs[k], stream)

    # end to end: pinned host inputs -> device -> kernel -> host, with E2E_BUFFERS device
    # buffer sets so that one step's copies overlap another step's kernel (e2e_pipeline).
    # A step's inputs (activations, letters, per-channel vectors) are packed into one
    # pinned host block and one device block per buffer set, so each step moves them in one
    # copy instead of eight (each copy has a fixed cost of several microseconds).
    def e2e_setup(self):
        torch = self.torch
        import numpy as np
        d = self.host
        parts = [("x", d["x"].view(np.uint8))]
        parts += [(k, d[k].view(np.uint8)) for k in ("wr", "wi", "wj", "wk")]
        parts += [(k, d[k].view(np.uint8)) for k in ("bias", "scale", "shift") if d[k] is not None]
        self.e2e_layout, off = {}, 0
        for name, a in parts:
            self.e2e_layout[name] = (off, a.nbytes)
            off += (a.nbytes + 255) // 256 * 256
        host = np.zeros(off, dtype=np.uint8)
        for name, a in parts:
            o, n = self.e2e_layout[name]
            host[o:o + n] = np.ascontiguousarray(a).reshape(-1)
        self.h_in = torch.from_numpy(host).pin_memory()
        s = self.spec
        out_bytes = s.N * s.Ho * s.Wo * s.Cout * 2
        self.h_out = [torch.empty(out_bytes, dtype=torch.uint8).pin_memory()
                      for _ in range(E2E_BUFFERS)]
        self.e_in = [torch.empty_like(self.h_in, device="cuda") for _ in range(E2E_BUFFERS)]
        self.e_out = [torch.empty_like(t, device="cuda") for t in self.h_out]
        self.h2d = sum(n for _, n in self.e2e_layout.values())
        self.d2h = out_bytes

    def e2e_in(self, b):
        return [(self.e_in[b], self.h_in)]

    def e2e_out(self, b):
        return [(self.h_out[b], self.e_out[b])]

    def e2e_compute(self, b, stream):
        torch, s, q = self.torch, self.spec, self.quan

        def view(name, dtype):
            if name not in self.e2e_layout:
                return None
            o, n = self.e2e_layout[name]
            return self.e_in[b][o:o + n].view(dtype)

        w = [view(k, torch.bfloat16) for k in ("wr", "wi", "wj", "wk")]
        out = self.e_out[b].view(torch.bfloat16).view(s.N, s.Ho, s.Wo, s.Cout)
        self.conv(view("x", torch.bfloat16), *w, view("bias", torch.float32),
                  view("scale", torch.float32), view("shift", torch.float32), s.N, s.H, s.W,
                  s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act, out, stream)

    @property
    def flops(self):
        # the separable form keeps the 4 diagonal component convolutions of the 16
        return self.spec.flops / 4 if self.separable else self.spec.flops

    @property
    def algorithmic_bytes(self):
        return self.spec.algorithmic_bytes


class BwdRunner:
    """Backward pass of one layer: dx (quan_qconv2d[_sep]_bwd_data) and dW
    (quan_qconv2d[_sep]_bwd_weight) from a seeded output gradient, with rotating buffer
    sets like LayerRunner."""

    def __init__(self, spec, torch, quan, inputs, separable=False):
        import numpy as np
        self.spec, self.torch, self.quan = spec, torch, quan
        self.separable = separable
        self.bwd_data = quan.quan_qconv2d_sep_bwd_data if separable else quan.quan_qconv2d_bwd_data
        self.bwd_weight = (quan.quan_qconv2d_sep_bwd_weight if separable
                           else quan.quan_qconv2d_bwd_weight)
        d = inputs.layer_inputs(spec)
        d["dy"] = inputs.grad_output(spec)
        dev = torch.device("cuda")

        def up(a):
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(
                torch.bfloat16).to(dev)

        self.host = d
        x0, dy0 = up(d["x"]), up(d["dy"])
        self.w = [up(d[k]) for k in ("wr", "wi", "wj", "wk")]
        per_set = (2 * x0.numel() + 2 * dy0.numel()) * 2  # x, dy read; dx written
        self.sets = max(2, min(16, math.ceil(2 * L2_BYTES / per_set)))
        self.xs = [x0] + [x0.clone() for _ in range(self.sets - 1)]
        self.dys = [dy0] + [dy0.clone() for _ in range(self.sets - 1)]
        self.dxs = [torch.empty_like(x0) for _ in range(self.sets)]
        wshape = (spec.Cout // 4, spec.kh, spec.kw, spec.Cin // 4)
        self.dws = [torch.empty(wshape, dtype=torch.float32, device=dev) for _ in range(4)]
        self.ws_bytes = quan.quan_qconv2d_bwd_data_workspace_size_ex(
            spec.N, spec.H, spec.W, spec.Cin, spec.Cout, spec.kh, spec.kw, spec.stride,
            spec.pad)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=dev)
        self.i = 0
        self.footprint = per_set * self.sets
        self.launches_per_step = None  # set by count_launches()

    def data(self, k, stream):
        s = self.spec
        self.bwd_data(self.dys[k], *self.w, s.N, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw, s.stride,
                      s.pad, self.ws, self.ws_bytes, self.dxs[k], stream)

    def weight(self, k, stream):
        s = self.spec
        self.bwd_weight(self.xs[k], self.dys[k], s.N, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw,
                        s.stride, s.pad, *self.dws, stream)

    def step(self, stream):
        k = self.i % self.sets
        self.i += 1
        self.data(k, stream)
        self.weight(k, stream)

    def count_launches(self, stream):
        """Kernels of this library one step launches (the tensor-core input gradient is a
        weight transform plus one convolution kernel; the weight gradient one kernel)."""
        self.data(0, stream)
        n = 2 if self.quan.quan_last_path() == self.quan.QUAN_PATH_TC else 1
        self.data_kernel = self.quan.quan_last_kernel()
        self.weight(0, stream)
        self.weight_kernel = self.quan.quan_last_kernel()
        self.launches_per_step = n + 1

    def e2e_setup(self):
        torch = self.torch
        import numpy as np
        d = self.host
        parts = [("x", d["x"].view(np.uint8)), ("dy", d["dy"].view(np.uint8))]
        parts += [(k, d[k].view(np.uint8)) for k in ("wr", "wi", "wj", "wk")]
        self.e2e_layout, off = {}, 0
        for name, a in parts:
            self.e2e_layout[name] = (off, a.nbytes)
            off += (a.nbytes + 255) // 256 * 256
        host = np.zeros(off, dtype=np.uint8)
        for name, a in parts:
            o, n = self.e2e_layout[name]
            host[o:o + n] = np.ascontiguousarray(a).reshape(-1)
        self.h_in = torch.from_numpy(host).pin_memory()
        s = self.spec
        dx_bytes = s.N * s.H * s.W * s.Cin * 2
        dw_bytes = s.Cout * s.Cin * s.kh * s.kw // 4 * 4  # four fp32 letters
        self.out_layout = (dx_bytes, (dx_bytes + 255) // 256 * 256)
        out_total = self.out_layout[1] + dw_bytes
        self.h_out = [torch.empty(out_total, dtype=torch.uint8).pin_memory()
                      for _ in range(E2E_BUFFERS)]
        self.e_in = [torch.empty_like(self.h_in, device="cuda") for _ in range(E2E_BUFFERS)]
        self.e_out = [torch.empty_like(t, device="cuda") for t in self.h_out]
        self.h2d = sum(n for _, n in self.e2e_layout.values())
        self.d2h = dx_bytes + dw_bytes

    def e2e_in(self, b):
        return [(self.e_in[b], self.h_in)]

    def e2e_out(self, b):
        return [(self.h_out[b], self.e_out[b])]

    def e2e_compute(self, b, stream):
        torch, s = self.torch, self.spec

        def view(name):
            o, n = self.e2e_layout[name]
            return self.e_in[b][o:o + n].view(torch.bfloat16)

        dx_bytes, dw_off = self.out_layout
        dx = self.e_out[b][:dx_bytes]
        per = s.Cout * s.Cin * s.kh * s.kw // 16 * 4
        dw = [self.e_out[b][dw_off + L * per:dw_off + (L + 1) * per].view(torch.float32)
              for L in range(4)]
        w = [view(k) for k in ("wr", "wi", "wj", "wk")]
        self.bwd_data(view("dy"), *w, s.N, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw, s.stride,
                      s.pad, self.ws, self.ws_bytes, dx, stream)
        self.bwd_weight(view("x"), view("dy"), s.N, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw,
                        s.stride, s.pad, *dw, stream)

    @property
    def flops(self):
        # input and weight gradients, each as many multiply-adds as the forward
        return 2 * self.spec.flops / (4 if self.separable else 1)

    def kernel_times(self, torch, stream, reps=5):
        """Average duration of the input-gradient and weight-gradient calls, timed apart
        with events on the launching stream (outside the timed region)."""
        sh = stream.cuda_stream
        out = []
        for fn in (self.data, self.weight):
            for k in range(2):
                fn(k % self.sets, sh)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for r in range(reps):
                fn(r % self.sets, sh)
            e1.record(stream)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) / reps / 1e3)
        return out


def bwd_roofline(runner, torch, stream, peaks, peak_src, direction_key):
    """Roofline of the slower of the two gradient calls.  Tensor-core input gradient:
    FLOPs against the bf16 peak; CUDA-core gradients: FLOPs against the fp32 FFMA peak
    (152 SMs x 128 lanes x 2 FLOP x 2.07 GHz maximum clock)."""
    t_data, t_weight = runner.kernel_times(torch, stream)
    half = runner.flops / 2
    rows = []
    for name, t, kernel in (("dx", t_data, runner.data_kernel),
                            ("dW", t_weight, runner.weight_kernel)):
        tc = kernel.startswith("qconv_")
        peak = peaks["bf16_tflops"] if tc else FP32_ALU_TFLOPS
        ach = half / t / 1e12
        rows.append({"grad": name, "kernel": kernel, "ms": round(t * 1e3, 4),
                     "bound": "tensor" if tc else "alu", "achieved": round(ach, 2),
                     "peak": peak, "frac": round(ach / peak, 4)})
    top = max(rows, key=lambda r: r["ms"])
    src = (peak_src + " (burst)" if top["bound"] == "tensor"
           else "derived: 152 SMs x 128 FP32 lanes x 2 FLOP x 2070 MHz")
    return {"bound": top["bound"], "achieved": top["achieved"], "peak": top["peak"],
            "unit": "TFLOP/s", "frac": top["frac"],
            "traffic": recorded_traffic(direction_key, top["kernel"]),
            "kernel": "%s (%s)" % (top["kernel"], top["grad"]),
            "share": round(top["ms"] / (rows[0]["ms"] + rows[1]["ms"]), 3),
            "peak_source": src, "algorithmic_flops": half, "gradients": rows}


def cpu_bwd_sample(spec, seconds, inputs, separable=False):
    """Time the fp64 oracle's two gradients on a bounded number of images."""
    import oracle
    d = inputs.layer_inputs(spec, n_images=1)
    f64 = oracle.bf16_bits_to_f64
    w = [f64(d[k]) for k in ("wr", "wi", "wj", "wk")]
    bd = oracle.qconv2d_sep_bwd_data if separable else oracle.qconv2d_bwd_data
    bw = oracle.qconv2d_sep_bwd_weight if separable else oracle.qconv2d_bwd_weight

    def run(n):
        x = f64(inputs.layer_inputs(spec, n_images=n)["x"])
        dy = f64(inputs.grad_output(spec, n_images=n))
        t0 = time.perf_counter()
        bd(dy, *w, H=spec.H, W=spec.W, stride=spec.stride, pad=spec.pad)
        bw(x, dy, kh=spec.kh, kw=spec.kw, stride=spec.stride, pad=spec.pad)
        return time.perf_counter() - t0

    t1 = run(1)
    n = max(1, min(spec.N, int(seconds / max(t1, 1e-6))))
    t = run(n) if n > 1 else t1
    flop = 2 * spec.flops / spec.N * n / (4 if separable else 1)
    return {"value": flop / t / 1e12, "unit": "TFLOP/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": "input and weight gradients of %d of %d images of the layer (fp64, "
                      "%.2f s)" % (n, spec.N, t)}


def cpu_oracle_sample(spec, seconds, inputs, separable=False):
    """Time the fp64 oracle on a bounded number of images of the layer."""
    import oracle
    d = inputs.layer_inputs(spec, n_images=1)
    f64 = oracle.bf16_bits_to_f64
    w = [f64(d[k]) for k in ("wr", "wi", "wj", "wk")]
    conv = oracle.qconv2d_separable if separable else oracle.qconv2d

    def run(n):
        dd = inputs.layer_inputs(spec, n_images=n)
        x = f64(dd["x"])
        t0 = time.perf_counter()
        conv(x, *w, stride=spec.stride, pad=spec.pad, bias=d["bias"], scale=d["scale"],
             shift=d["shift"], act=spec.act)
        return time.perf_counter() - t0

    t1 = run(1)
    n = max(1, min(spec.N, int(seconds / max(t1, 1e-6))))
    t = run(n) if n > 1 else t1
    flop = spec.flops / spec.N * n / (4 if separable else 1)
    return {"value": flop / t / 1e12, "unit": "TFLOP/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": "%d of %d images of the layer (fp64, %.2f s)" % (n, spec.N, t)}


# ---------------------------------------------------------------------------- main

WORKLOAD_DESC = {
    "c1": "CIFAR-shaped QUAN layer",
    "c2a": "ImageNet ResNet-stage layer",
    "c2b": "ImageNet ResNet-stage stride-2 layer",
    "c3a": "detection-neck pointwise layer",
    "c3b": "detection-neck 3x3 layer",
    "backbone": "ResNet-18-style QUAN backbone",
    "poincare": "Poincare RGB -> quaternion input mapping (Eq. 4)",
    "iqbn": "training-mode IQBN (Eq. 11-12): batch statistics, then normalisation + ReLU",
}

POINCARE_SHAPE = (256, 224, 224)  # the backbone's input batch: N, H, W
IQBN_SHAPE = (64, 56, 56, 256)    # the ImageNet-stage layer's output: N, H, W, C


class IqbnRunner:
    """Training-mode IQBN of one activation tensor (bf16 NHWC): quan_iqbn_batch_stats, then
    quan_iqbn_train_fwd with ReLU into a separate output, on rotating buffer sets larger
    than L2."""

    def __init__(self, torch, quan, inputs, N, H, W, C):
        import numpy as np
        self.torch, self.quan, self.N, self.C = torch, quan, N, C
        self.npix = N * H * W
        rng = np.random.default_rng(45)
        x = rng.standard_normal((N, H, W, C), dtype=np.float32) + np.float32(0.5)
        self.host_x = inputs.to_bf16_bits(x)
        self.host_gamma = rng.uniform(0.5, 1.5, C).astype(np.float32)
        self.host_beta = (rng.standard_normal(C, dtype=np.float32) * np.float32(0.1))
        x0 = torch.from_numpy(self.host_x.view(np.int16)).view(torch.bfloat16).cuda()
        per_set = self.npix * C * 4  # x and out
        self.sets = max(2, min(8, math.ceil(2 * L2_BYTES / per_set)))
        self.xs = [x0] + [x0.clone() for _ in range(self.sets - 1)]
        self.outs = [torch.empty_like(x0) for _ in range(self.sets)]
        self.gamma = torch.from_numpy(self.host_gamma).cuda()
        self.beta = torch.from_numpy(self.host_beta).cuda()
        self.mean = torch.empty(C, dtype=torch.float32, device="cuda")
        self.var = torch.empty(C, dtype=torch.float32, device="cuda")
        self.ws_bytes = quan.quan_iqbn_batch_stats_workspace_size(C)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device="cuda")
        self.i = 0
        self.launches_per_step = 3  # statistics, finalisation, normalisation
        self.footprint = per_set * self.sets
        self.flops = 0.0
        self.stats_bytes = float(self.npix * C * 2)      # x read once
        self.apply_bytes = float(self.npix * C * 4)      # x read, out written
        self.algorithmic_bytes = self.stats_bytes + self.apply_bytes
        self.separable = False

    def stats(self, k, stream):
        self.quan.quan_iqbn_batch_stats(self.xs[k], self.npix, self.C, self.ws, self.ws_bytes,
                                        self.mean, self.var, stream)

    def apply(self, k, stream):
        self.quan.quan_iqbn_train_fwd(self.xs[k], self.npix, self.C, self.mean, self.var,
                                      self.gamma, self.beta, 1e-5, self.quan.QUAN_ACT_RELU,
                                      self.outs[k], stream)

    def step(self, stream):
        k = self.i % self.sets
        self.i += 1
        self.stats(k, stream)
        self.apply(k, stream)

    def kernel_times(self, torch, stream, reps=5):
        sh = stream.cuda_stream
        out = []
        for fn in (self.stats, self.apply):
            for k in range(2):
                fn(k % self.sets, sh)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for r in range(reps):
                fn(r % self.sets, sh)
            e1.record(stream)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) / reps / 1e3)
        return out

    def e2e_setup(self):
        torch = self.torch
        import numpy as np
        self.h_in = torch.from_numpy(self.host_x.view(np.int16).reshape(-1)).pin_memory()
        self.h_out = [torch.empty(self.npix * self.C, dtype=torch.int16).pin_memory()
                      for _ in range(E2E_BUFFERS)]
        self.e_in = [torch.empty_like(self.h_in, device="cuda") for _ in range(E2E_BUFFERS)]
        self.e_out = [torch.empty_like(t, device="cuda") for t in self.h_out]
        self.h2d = self.npix * self.C * 2
        self.d2h = self.npix * self.C * 2

    def e2e_in(self, b):
        return [(self.e_in[b], self.h_in)]

    def e2e_out(self, b):
        return [(self.h_out[b], self.e_out[b])]

    def e2e_compute(self, b, stream):
        q = self.quan
        q.quan_iqbn_batch_stats(self.e_in[b], self.npix, self.C, self.ws, self.ws_bytes,
                                self.mean, self.var, stream)
        q.quan_iqbn_train_fwd(self.e_in[b], self.npix, self.C, self.mean, self.var, self.gamma,
                              self.beta, 1e-5, q.QUAN_ACT_RELU, self.e_out[b], stream)


def iqbn_roofline(runner, torch, stream, peaks, peak_src):
    """HBM roofline of the slower of the two kernels, timed apart with events."""
    t_stats, t_apply = runner.kernel_times(torch, stream)
    rows = [{"kernel": "iqbn_stats_kernel (+ finalize)", "ms": round(t_stats * 1e3, 4),
             "achieved": round(runner.stats_bytes / t_stats / 1e9, 1)},
            {"kernel": "iqbn_apply_kernel", "ms": round(t_apply * 1e3, 4),
             "achieved": round(runner.apply_bytes / t_apply / 1e9, 1)}]
    for r in rows:
        r["frac"] = round(r["achieved"] / peaks["hbm_gbs"], 4)
    top = max(rows, key=lambda r: r["ms"])
    return {"bound": "hbm", "achieved": top["achieved"], "peak": peaks["hbm_gbs"],
            "unit": "GB/s", "frac": top["frac"],
            "traffic": recorded_traffic("iqbn", top["kernel"].split()[0]),
            "kernel": top["kernel"], "share": round(top["ms"] / (rows[0]["ms"] + rows[1]["ms"]), 3),
            "peak_source": peak_src + " (burst)", "kernels": rows}


def iqbn_cpu_sample(runner, seconds):
    """The fp64 oracle's training-mode IQBN on a bounded number of images of the batch."""
    import oracle
    f64 = oracle.bf16_bits_to_f64
    g, b = runner.host_gamma.astype("float64"), runner.host_beta.astype("float64")
    t0 = time.perf_counter()
    oracle.iqbn_train(f64(runner.host_x[:1]), g, b, act=oracle.ACT_RELU)
    t1 = max(time.perf_counter() - t0, 1e-6)
    n = max(1, min(runner.N, int(seconds / t1)))
    x = f64(runner.host_x[:n])
    t0 = time.perf_counter()
    oracle.iqbn_train(x, g, b, act=oracle.ACT_RELU)
    t = time.perf_counter() - t0
    return {"value": n / t, "unit": "images/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": "statistics and normalisation of %d of %d images of the batch (fp64, "
                      "%.2f s)" % (n, runner.N, t)}


class PoincareRunner:
    """The Eq. 4 input mapping of an image batch, fp32 RGB -> bf16 quaternion pixels, on
    rotating buffer sets larger than L2."""

    def __init__(self, torch, quan, N, H, W):
        import numpy as np
        self.torch, self.quan, self.N = torch, quan, N
        self.npix = N * H * W
        rng = np.random.default_rng(44)
        self.host_rgb = rng.uniform(0.0, 1.0, size=(N, H, W, 3)).astype(np.float32)
        rgb0 = torch.from_numpy(self.host_rgb).cuda()
        per_set = self.npix * 20
        self.sets = max(2, min(8, math.ceil(2 * L2_BYTES / per_set)))
        self.rgb = [rgb0] + [rgb0.clone() for _ in range(self.sets - 1)]
        self.out = [torch.empty((N, H, W, 4), dtype=torch.bfloat16, device="cuda")
                    for _ in range(self.sets)]
        self.i = 0
        self.launches_per_step = 1
        self.footprint = per_set * self.sets
        self.flops = 0.0
        self.algorithmic_bytes = float(per_set)  # 12 bytes read, 8 written per pixel
        self.separable = False

    def step(self, stream):
        k = self.i % self.sets
        self.i += 1
        self.quan.quan_poincare_fwd(self.rgb[k], self.npix, self.out[k], stream)

    def e2e_setup(self):
        torch = self.torch
        self.h_in = torch.from_numpy(self.host_rgb.reshape(-1)).pin_memory()
        self.h_out = [torch.empty(self.npix * 4, dtype=torch.bfloat16).pin_memory()
                      for _ in range(E2E_BUFFERS)]
        self.e_in = [torch.empty_like(self.h_in, device="cuda") for _ in range(E2E_BUFFERS)]
        self.e_out = [torch.empty_like(t, device="cuda") for t in self.h_out]
        self.h2d = self.npix * 12
        self.d2h = self.npix * 8

    def e2e_in(self, b):
        return [(self.e_in[b], self.h_in)]

    def e2e_out(self, b):
        return [(self.h_out[b], self.e_out[b])]

    def e2e_compute(self, b, stream):
        self.quan.quan_poincare_fwd(self.e_in[b], self.npix, self.e_out[b], stream)


def poincare_cpu_sample(runner, seconds):
    """Time the fp64 oracle mapping on a bounded number of images of the batch."""
    import numpy as np
    import oracle
    img = runner.host_rgb[0].astype(np.float64)
    t0 = time.perf_counter()
    oracle.poincare(img)
    t1 = max(time.perf_counter() - t0, 1e-6)
    n = max(1, min(runner.N, int(seconds / t1)))
    t0 = time.perf_counter()
    for i in range(n):
        oracle.poincare(runner.host_rgb[i].astype(np.float64))
    t = time.perf_counter() - t0
    return {"value": n / t, "unit": "images/s", "cores": 1, "kind": "oracle",
            "sample": "%d of %d images of the batch (fp64, %.2f s)" % (n, runner.N, t)}


def act_code(name: str) -> int:
    return {"relu": 1, "silu": 2}[name]


def workload_config(workload: str, inputs, variant: str = "full", direction: str = "fwd",
                    act: str = "relu", rgb: bool = False) -> dict:
    """The workload part of the JSON line's config, shared by both arms."""
    if workload == "poincare":
        N, H, W = POINCARE_SHAPE
        return {"workload": "%s, N=%d, %dx%d fp32 RGB -> bf16 quaternion pixels" % (
                    WORKLOAD_DESC[workload], N, H, W), "N": N, "H": H, "W": W,
                "bytes_per_step": N * H * W * 20}
    if workload == "iqbn":
        N, H, W, C = IQBN_SHAPE
        return {"workload": "%s, N=%d, %dx%d, C=%d bf16" % (WORKLOAD_DESC[workload], N, H, W, C),
                "N": N, "H": H, "W": W, "C": C, "bytes_per_step": N * H * W * C * 6}
    if workload == "backbone":
        layers = inputs.backbone_layers(act=act_code(act))
        convs = [L.spec for L in layers if L.kind == "conv"]
        c0 = convs[0]
        return {"workload": "%s, N=%d, %dx%d%s" % (
                    WORKLOAD_DESC[workload], c0.N, c0.H, c0.W,
                    " fp32 RGB input (Eq. 4 mapping in the stem kernel's loader)" if rgb
                    else "x4 quaternion input"),
                "N": c0.N, "H": c0.H, "W": c0.W, "convs": len(convs), "maxpool": 1,
                "flops_per_step": sum(c.flops for c in convs),
                "epilogue": "IQBN+%s (+residual)" % ("SiLU" if act == "silu" else "ReLU"),
                "fusions": "stem conv + 3x3/2 max pool in one kernel (only the pooled tensor is written)"}
    s = inputs.LAYERS[workload]
    cfg = {"workload": WORKLOAD_DESC[workload], "N": s.N, "H": s.H, "W": s.W, "Cin": s.Cin,
           "Cout": s.Cout, "kernel": "%dx%d" % (s.kh, s.kw), "stride": s.stride, "pad": s.pad,
           "epilogue": "IQBN+ReLU", "flops_per_step": s.flops}
    if variant == "separable":
        cfg["workload"] += ", separable form (Eq. 7)"
        cfg["flops_per_step"] = s.flops / 4
    if direction == "bwd":
        cfg["workload"] += ", backward: input and weight gradients before the epilogue" + (
            " (Eq. 8-10)" if variant == "separable" else "")
        cfg["flops_per_step"] *= 2
        cfg["epilogue"] = "none (gradient of the convolution's accumulator)"
    return cfg


def max_over_ranks(ms: float, dist, torch, device: str) -> float:
    """Slowest rank's time: every rank runs the same replica workload, the job ends when
    the last one does.  No-op without a process group."""
    if dist is None:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_step: float, steps: int, world: int, ms: float) -> float:
    """Whole-job rate: every rank processes units_per_step per step (weak scaling)."""
    return units_per_step * steps * world / (ms / 1e3)


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    from paper_2509_05512_gb300 import inputs

    if args.impl == "reference":
        return reference_arm(args, rank, world, inputs)

    import torch
    from paper_2509_05512_gb300 import build, quan

    torch.cuda.set_device(local_rank)
    build.build_library()
    quan.load()
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))

    def barrier():
        if dist is not None:
            dist.barrier()

    if args.batch and not args.profile:
        raise SystemExit("--batch is for --profile runs only")
    if args.workload in ("backbone", "poincare", "iqbn") and (args.variant != "full" or
                                                       args.direction != "fwd"):
        raise SystemExit("--variant and --pass apply to the convolution layer workloads")
    if args.workload != "backbone" and (args.act != "relu" or args.rgb):
        raise SystemExit("--act and --rgb apply to the backbone workload")
    if args.rgb and args.no_fuse:
        raise SystemExit("--rgb needs the fused stem")
    if args.workload == "poincare":
        runner = PoincareRunner(torch, quan, *POINCARE_SHAPE)
        unit, per_step_units, dtype = "images/s", runner.N, "f32->bf16"
    elif args.workload == "iqbn":
        runner = IqbnRunner(torch, quan, inputs, *IQBN_SHAPE)
        unit, per_step_units, dtype = "images/s", runner.N, "bf16 (fp32 statistics)"
    elif args.workload == "backbone":
        from paper_2509_05512_gb300 import backbone
        runner = backbone.BackboneRunner(torch, quan, inputs, N=args.batch or 256,
                                         act=act_code(args.act),
                                         fuse_stem_pool=not args.no_fuse, rgb=args.rgb,
                                         overlap_shortcuts=not args.no_overlap,
                                         split_k=not args.no_split)
        runner.sets = 1
        unit, per_step_units, dtype = "images/s", runner.N, "bf16"
    else:
        spec = inputs.LAYERS[args.workload]
        if args.batch:
            import dataclasses
            spec = dataclasses.replace(spec, N=args.batch)
        cls = BwdRunner if args.direction == "bwd" else LayerRunner
        runner = cls(spec, torch, quan, inputs, separable=args.variant == "separable")
        if args.direction == "bwd":
            runner.count_launches(torch.cuda.current_stream().cuda_stream)
        unit, per_step_units, dtype = "TFLOP/s", runner.flops / 1e12, "bf16"
    stream = torch.cuda.current_stream()
    sh = stream.cuda_stream

    if args.profile:
        for _ in range(args.warmup + args.steps):
            runner.step(sh)
        torch.cuda.synchronize()
        st, bits = quan.quan_device_status(sh)
        print(json.dumps({"profile_run": args.workload, "launches": args.warmup + args.steps,
                          "status": st}))
        return 0 if st == quan.QUAN_OK else 1

    # warm-up: at least W steps, and enough untimed steps for the clocks to settle
    gpu_id = getattr(torch.cuda.get_device_properties(local_rank), "uuid", None)
    gpu_id = ("GPU-" + str(gpu_id)) if gpu_id is not None else str(local_rank)
    sampler = ClockSampler(gpu_id) if rank == 0 else None
    t_end = time.perf_counter() + 1.0
    n = 0
    while n < args.warmup or time.perf_counter() < t_end:
        runner.step(sh)
        n += 1
        if n % 64 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    kernel_name = (None if args.workload in ("backbone", "iqbn") else
                   "poincare_kernel" if args.workload == "poincare" else quan.quan_last_kernel())

    # The timed region is exactly K steps.  By default they are captured once into a CUDA
    # graph (same launches, same buffers) so host launch overhead does not leave gaps.
    graph = None
    if not args.no_graph:
        cap = torch.cuda.Stream()
        cap.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=cap):
            for _ in range(args.steps):
                runner.step(cap.cuda_stream)
        torch.cuda.synchronize()
        graph.replay()  # warm replay (untimed)
        torch.cuda.synchronize()

    barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    if graph is not None:
        graph.replay()
    else:
        for _ in range(args.steps):
            runner.step(sh)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = ev0.elapsed_time(ev1)
    clocks = sampler.stop() if sampler else None
    ms = max_over_ranks(ms, dist, torch, "cuda")
    st, bits = quan.quan_device_status(sh)
    if st != quan.QUAN_OK:
        raise RuntimeError("kernel reported a timeout (bits 0x%x)" % bits)
    ms_per_step = ms / args.steps
    value = job_throughput(per_step_units, args.steps, world, ms)

    # end to end through the public call with host buffers
    e2e = None
    if not args.no_e2e:
        runner.e2e_setup()
        e2e_pipeline(runner, torch, stream, max(3, args.warmup))
        torch.cuda.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        e2e_pipeline(runner, torch, stream, args.steps)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ems = max_over_ranks(e0.elapsed_time(e1), dist, torch, "cuda")
        e2e = {"value": job_throughput(per_step_units, args.steps, world, ems), "unit": unit,
               "h2d_bytes_per_step": int(runner.h2d), "d2h_bytes_per_step": int(runner.d2h)}

    peaks, peak_src = load_peaks()
    if args.workload == "backbone":
        roofline = backbone_roofline(runner, torch, stream, peaks, peak_src)
    elif args.workload == "iqbn":
        roofline = iqbn_roofline(runner, torch, stream, peaks, peak_src)
    elif args.direction == "bwd":
        roofline = bwd_roofline(runner, torch, stream, peaks, peak_src, traffic_key(args))
    else:
        roofline = runner_roofline(runner, args, ms_per_step, peaks, peak_src, kernel_name)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        if args.workload == "backbone":
            cpu = backbone_cpu_sample(runner, args.cpu_seconds, inputs)
        elif args.workload == "poincare":
            cpu = poincare_cpu_sample(runner, args.cpu_seconds)
        elif args.workload == "iqbn":
            cpu = iqbn_cpu_sample(runner, args.cpu_seconds)
        elif args.direction == "bwd":
            cpu = cpu_bwd_sample(runner.spec, args.cpu_seconds, inputs,
                                 separable=runner.separable)
        else:
            cpu = cpu_oracle_sample(runner.spec, args.cpu_seconds, inputs,
                                    separable=runner.separable)

    if dist is not None:
        dist.destroy_process_group()
    if rank != 0:
        return 0
    cfg = workload_config(args.workload, inputs, args.variant, args.direction, args.act,
                          args.rgb)
    cfg.update({"l2": "inputs larger than L2: %d rotating buffer sets, %.0f MB" % (
                    getattr(runner, "sets", 1), runner.footprint / 1e6),
                "parallelism": "replicas over the batch (dp%d, no collective)" % world,
                "timing": "one CUDA-graph replay of the K steps" if graph is not None
                else "plain launch loop"})
    if args.workload == "backbone" and not getattr(runner, "fused", False):
        cfg["fusions"] = "none"
    if args.workload == "backbone":
        cfg["streams"] = ("the 1x1/2 shortcuts on a second stream beside their block's 3x3/2 "
                          "convolution" if getattr(runner, "side", None) else "one stream")
        cfg["split_k"] = getattr(runner, "workspace", None) is not None
    if args.workload not in ("backbone", "poincare", "iqbn") and args.direction == "fwd":
        cfg["path"] = {1: "tc", 2: "simt"}.get(quan.quan_last_path(), "?")
    if args.direction == "bwd":
        cfg["kernels"] = {"dx": runner.data_kernel, "dW": runner.weight_kernel}
    line = {"metric": METRIC, "value": round(value, 4), "unit": unit, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": dtype,
            "data": "synthetic (seeded; shapes of the paper's workloads)", "config": cfg,
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": runner.launches_per_step * args.steps, "clocks": clocks}
    print(json.dumps(line))
    return 0


def traffic_key(args) -> str:
    """Key of the workload in the recorded ncu traffic table."""
    return (args.workload + (":bwd" if args.direction == "bwd" else "") +
            (":sep" if args.variant == "separable" else ""))


def runner_roofline(runner, args, ms_per_step, peaks, peak_src, kernel_name):
    flops, nbytes = runner.flops, runner.algorithmic_bytes
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    t = ms_per_step / 1e3  # one kernel launch per step
    if flops / nbytes >= ridge:
        achieved, peak, unit, bound = flops / t / 1e12, peaks["bf16_tflops"], "TFLOP/s", "tensor"
    else:
        achieved, peak, unit, bound = nbytes / t / 1e9, peaks["hbm_gbs"], "GB/s", "hbm"
    return {"bound": bound, "achieved": round(achieved, 2), "peak": peak, "unit": unit,
            "frac": round(achieved / peak, 4),
            "traffic": recorded_traffic(traffic_key(args), kernel_name),
            "kernel": kernel_name, "peak_source": peak_src + " (burst)",
            "algorithmic_flops": flops, "algorithmic_bytes": nbytes}


def backbone_roofline(runner, torch, stream, peaks, peak_src):
    """Time every layer once with events on the launching stream (outside the timed
    region), then report the roofline of the layer with the largest share of the step."""
    sh = stream.cuda_stream
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    times, kernels = [], []
    for i, L in enumerate(runner.layers):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for _ in range(2):
            runner.run_layer(i, sh, workspace=getattr(runner, "workspace", None))
        kernels.append(runner.quan.quan_last_kernel() if L.kind == "conv" else "maxpool_kernel")
        e0.record(stream)
        for _ in range(5):
            runner.run_layer(i, sh, workspace=getattr(runner, "workspace", None))
        e1.record(stream)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) / 5 / 1e3)
    layers = []
    fused = getattr(runner, "fused", False)
    for i, (L, t) in enumerate(zip(runner.layers, times)):
        if fused and L.kind == "maxpool" and L.src == 0:
            continue  # part of the stem's fused call (layer 0)
        if L.kind == "conv":
            fl, nb = L.spec.flops, L.spec.algorithmic_bytes
            if L.res is not None:
                nb += L.spec.N * L.spec.Ho * L.spec.Wo * L.spec.Cout * 2
            name = "conv%dx%d/%d %d->%d @%d" % (L.spec.kh, L.spec.kw, L.spec.stride, L.spec.Cin,
                                                L.spec.Cout, L.spec.H)
            if fused and i == 0:
                # stem + 3x3/2 max pool: the pooled output replaces the stem's
                s0 = L.spec
                nb += (runner.outs[1].numel() - s0.N * s0.Ho * s0.Wo * s0.Cout) * 2
                name += " + maxpool3/2 (fused)"
                if getattr(runner, "rgb", False):  # 12 bytes of RGB per pixel, not 8
                    nb += s0.N * s0.H * s0.W * 4
                    name = "poincare (Eq. 4) + " + name
        else:
            src = runner.outs[L.src]
            fl, nb = 0.0, src.numel() * 2 + runner.outs[i].numel() * 2
            name = "maxpool%d/%d" % (L.k, L.stride)
        bound = "tensor" if fl / nb >= ridge else "hbm"
        ach = fl / t / 1e12 if bound == "tensor" else nb / t / 1e9
        peak = peaks["bf16_tflops"] if bound == "tensor" else peaks["hbm_gbs"]
        layers.append({"layer": i, "name": name, "kernel": kernels[i], "ms": round(t * 1e3, 4),
                       "bound": bound, "achieved": round(ach, 1), "frac": round(ach / peak, 3)})
    top = max(layers, key=lambda r: r["ms"])
    total = sum(r["ms"] for r in layers)
    L = runner.layers[top["layer"]]
    fl = L.spec.flops if L.kind == "conv" else 0.0
    return {"bound": top["bound"], "achieved": top["achieved"],
            "peak": peaks["bf16_tflops"] if top["bound"] == "tensor" else peaks["hbm_gbs"],
            "unit": "TFLOP/s" if top["bound"] == "tensor" else "GB/s", "frac": top["frac"],
            "traffic": recorded_traffic("backbone", top["kernel"]),
            "kernel": "%s (%s)" % (top["kernel"], top["name"]),
            "share": round(top["ms"] / total, 3), "peak_source": peak_src + " (burst)",
            "layers": layers}


def backbone_cpu_sample(runner, seconds, inputs):
    """The fp64 oracle backbone on a bounded number of images (RGB input: the Eq. 4 mapping
    first, rounded to bf16 as the stem kernel's loader stores it, inside the timing)."""
    import numpy as np
    import oracle
    import oracle.backbone as ob
    params = [inputs.backbone_params(L) if L.kind == "conv" else None for L in runner.layers]
    rgb = getattr(runner, "rgb", False)

    def run(n):
        x = runner.x_host[:n]
        if rgb:
            x = inputs.to_bf16_bits(oracle.poincare(x.astype(np.float64)).astype(np.float32))
        ob.forward(inputs.backbone_layers(N=n, H=runner.H, act=runner.act), params, x)

    t0 = time.perf_counter()
    run(1)
    t1 = time.perf_counter() - t0
    n = max(1, min(runner.N, int(seconds / max(t1, 1e-6))))
    if n > 1:
        t0 = time.perf_counter()
        run(n)
        t1 = time.perf_counter() - t0
    return {"value": n / t1, "unit": "images/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": "%d of %d images of the backbone (fp64%s, %.2f s)" % (
                n, runner.N, ", from RGB" if rgb else "", t1)}


def reference_arm(args, rank, world, inputs):
    """The fp64 CPU oracle as the reference arm: each step is a bounded sample of the
    same workload (rank 0 only)."""
    if rank != 0:
        return 0
    import oracle
    ref_cfg = workload_config(args.workload, inputs, args.variant, args.direction, args.act,
                              args.rgb)
    ref_cfg["parallelism"] = "fp64 oracle on %d host threads" % oracle.num_threads()
    if args.workload == "poincare":
        import numpy as np
        N, H, W = POINCARE_SHAPE
        img = np.random.default_rng(44).uniform(0.0, 1.0, size=(H, W, 3))
        for _ in range(args.warmup):
            oracle.poincare(img)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            oracle.poincare(img)
        dt = time.perf_counter() - t0
        value = args.steps / dt
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "images/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": ref_cfg,
                "cpu_baseline": {"value": value, "unit": "images/s", "cores": 1,
                                 "kind": "oracle",
                                 "sample": "1 of %d images of the batch per step (fp64)" % N},
                "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0
    if args.workload == "iqbn":
        N, H, W, C = IQBN_SHAPE
        import numpy as np
        rng = np.random.default_rng(45)
        x = rng.standard_normal((1, H, W, C)) + 0.5
        g, b = rng.uniform(0.5, 1.5, C), rng.standard_normal(C) * 0.1
        for _ in range(args.warmup):
            oracle.iqbn_train(x, g, b, act=oracle.ACT_RELU)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            oracle.iqbn_train(x, g, b, act=oracle.ACT_RELU)
        dt = time.perf_counter() - t0
        value = args.steps / dt
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "images/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": ref_cfg,
                "cpu_baseline": {"value": value, "unit": "images/s",
                                 "cores": oracle.num_threads(), "kind": "oracle",
                                 "sample": "1 of %d images of the batch per step (fp64)" % N},
                "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0
    if args.workload == "backbone":
        import oracle.backbone as ob
        import numpy as np
        layers = inputs.backbone_layers(N=1, act=act_code(args.act))
        params = [inputs.backbone_params(L) if L.kind == "conv" else None for L in layers]
        x = inputs.backbone_input(n_images=1)
        rgb = inputs.backbone_rgb(n_images=1) if args.rgb else None

        def step():
            xs = x
            if rgb is not None:  # Eq. 4, rounded to bf16 as the stem kernel stores it
                xs = inputs.to_bf16_bits(
                    oracle.poincare(rgb.astype(np.float64)).astype(np.float32))
            ob.forward(layers, params, xs)

        for _ in range(args.warmup):
            step()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            step()
        dt = time.perf_counter() - t0
        value = args.steps / dt
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "images/s",
                "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": ref_cfg,
                "cpu_baseline": {"value": value, "unit": "images/s", "cores": oracle.num_threads(),
                                 "kind": "oracle",
                                 "sample": "1 of 256 images of the backbone per step (fp64)"},
                "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0
    spec = inputs.LAYERS[args.workload]
    d = inputs.layer_inputs(spec, n_images=1)
    f64 = oracle.bf16_bits_to_f64
    x = f64(d["x"])
    w = [f64(d[k]) for k in ("wr", "wi", "wj", "wk")]

    sep = args.variant == "separable"
    conv = oracle.qconv2d_separable if sep else oracle.qconv2d
    bwd = args.direction == "bwd"
    if bwd:
        dy = f64(inputs.grad_output(spec, n_images=1))
        bd = oracle.qconv2d_sep_bwd_data if sep else oracle.qconv2d_bwd_data
        bw = oracle.qconv2d_sep_bwd_weight if sep else oracle.qconv2d_bwd_weight

    def step():
        if bwd:
            bd(dy, *w, H=spec.H, W=spec.W, stride=spec.stride, pad=spec.pad)
            bw(x, dy, kh=spec.kh, kw=spec.kw, stride=spec.stride, pad=spec.pad)
            return
        conv(x, *w, stride=spec.stride, pad=spec.pad, bias=d["bias"], scale=d["scale"],
             shift=d["shift"], act=spec.act)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    per_step = spec.flops / spec.N / (4 if sep else 1) * (2 if bwd else 1)  # one image
    value = per_step * args.steps / dt / 1e12
    cpu = {"value": value, "unit": "TFLOP/s", "cores": oracle.num_threads(), "kind": "oracle",
           "sample": "1 of %d images of the layer per step (fp64%s)" % (
               spec.N, ", input and weight gradients" if bwd else "")}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": ref_cfg,
            "cpu_baseline": cpu,
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


if __name__ == "__main__":
    sys.exit(main())
