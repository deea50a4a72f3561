#!/usr/bin/env python
"""Skip-Conv layer-step benchmark on GB300.

Workload (one "step" = one Skip-Conv layer step over one batch):
  3x3 Skip-Conv layer, 256 -> 256 channels, 8 independent streams of 128x128
  frames, bf16 storage with fp32 accumulation, 8x8 gate blocks, eps 0.05,
  Input-Norm gate (mean over the support), with exactly 10% of the blocks of
  every stream changing per frame (synthetic video, seeded).

Reports stream-frames/s (value), effective TFLOP/s on the active locations,
the step's roofline fraction, the dominant kernel's roofline, an end-to-end
number through the host-buffer ABI call, the CPU oracle on the host cores,
and a density sweep against the library's all-ones dense mode.

    python bench.py [--steps K] [--warmup W] [--impl ours|reference] [--no-sweep]
Under torchrun every rank runs an independent replica (weak scaling).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Skip-Conv frames/s and effective TFLOP/s vs roofline at measured gate density"
UNIT = "stream-frames/s"
N_STREAMS, H, W, C, K, BLOCK, EPS = 8, 128, 128, 256, 3, 8, 0.05
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNELS = ("gate_pixel", "gate_block", "conv", "y_refresh", "step_fused", "step_local")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--density", type=float, default=0.10)
    ap.add_argument("--gate", choices=("input", "output", "gumbel"), default="input",
                    help="input: Input-Norm gate (Eq. 5, mean over the support); output: Output-Norm gate (Eq. 7); "
                         "gumbel: the Gumbel gate at inference (Eq. 8) with a seeded random phi (separate launches)")
    ap.add_argument("--key-interval", type=int, default=0,
                    help="a key frame every K steps (Table 4's periodic reset); 0: none after the first")
    ap.add_argument("--drift", action="store_true",
                    help="add a drift report: Skip-Conv z~ against the dense closed form for several key intervals")
    ap.add_argument("--path", choices=("fused", "separate"), default="fused",
                    help="fused: one launch per step (default); separate: gate passes and convolution launched apart")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--sweep-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the single-layer and stacked workloads (c0-c3)")
    ap.add_argument("--link", choices=("both", "on", "off"), default="both",
                    help="stack propagation for the stacked workloads: also time linked stacks (both), "
                         "link them throughout (on), or not at all (off)")
    ap.add_argument("--workloads-only", default=None, metavar="NAMES",
                    help="run only these of the single-layer and stacked workloads (comma-separated, e.g. c2,c3; "
                         "\"warped\" for the warped-residual pan) "
                         "and print their report; for profiling them")
    ap.add_argument("--no-flush", action="store_true",
                    help="no L2 flush between timed steps: each step streams 134 MB of frames, more than the L2")
    ap.add_argument("--no-soak", action="store_true",
                    help="skip the untimed steps around the timed region (for profiler runs)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-table", action="store_true",
                    help="skip the oracle's per-workload table (every config, all cores and one)")
    ap.add_argument("--cpu-table-seconds", type=float, default=1.5,
                    help="seconds of oracle work per row of the per-workload table")
    ap.add_argument("--clocks-log", default=None, metavar="PATH",
                    help="keep the nvidia-smi samples of the timed region in this CSV (default: a temporary file)")
    return ap.parse_args()


def workload_config(density, flushed=True, gate="input", key_interval=0):
    return {"workload": "c4: 3x3 Skip-Conv 256->256, %d streams x %dx%d, bf16 (fp32 accum), %dx%d blocks, "
                        "eps %.2g, %g%% block density" % (N_STREAMS, H, W, BLOCK, BLOCK, EPS, density * 100),
            "streams": N_STREAMS, "h": H, "w": W, "c_in": C, "c_out": C, "k": K, "block": BLOCK, "eps": EPS,
            "gate": {"input": "input-norm (mean over support)", "output": "output-norm (Eq. 7)",
                     "gumbel": "gumbel at inference (Eq. 8), f(r; phi) > eps, phi ~ N(0, 1/(9 c_in)) seeded, bias 0"}[gate],
            "key_interval": key_interval, "density": density,
            "l2": ("flushed between timed steps (256 MiB written, then read back)" if flushed else
                   "not flushed: each step streams two 64 MiB frames per step in stream order, more than the 129 MB L2"),
            "parallelism": "replicas"}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return d, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------- clocks
class Clocks:
    """nvidia-smi sampling during the timed regions."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index, path=None):
        self.index, self.proc, self.path = index, None, path

    def start(self):
        try:
            if self.path is None:
                import tempfile
                fd, self.path = tempfile.mkstemp(prefix="clocks_bench_", suffix=".csv")
                os.close(fd)
            else:
                os.makedirs(os.path.dirname(os.path.abspath(self.path)), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(5)
        except Exception:
            self.proc.kill()
        self.f.close()
        with open(self.path) as f:
            return self.summarise(f)

    @staticmethod
    def summarise(lines):
        """Median and maximum SM clock, maximum power and the throttle reasons seen active, from
        nvidia-smi's csv,noheader,nounits lines of the query Q (lines it could not measure are skipped)."""
        sm, smax, reasons, power = [], [], set(), []
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                clk, clk_max = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            sm.append(clk)
            smax.append(clk_max)
            try:
                power.append(float(parts[3]))
            except ValueError:
                pass
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None, "samples": len(sm), "reasons": sorted(reasons)}


# ------------------------------------------------------------- workloads
def device_frames(density, n_frames, rank, torch):
    import synth
    wl = synth.make_workload("c4", density=density, T=n_frames, n=N_STREAMS, h=H, w=W, c=C, block=BLOCK,
                             stream_offset=rank * N_STREAMS)
    frames, changed = [], []
    prev = None
    for t, f in wl.frames:
        x = torch.from_numpy(f).cuda().to(torch.bfloat16)        # bf16-exact values: no rounding
        if prev is not None:
            changed.append(int((x != prev).any(dim=-1).sum().item()))
        frames.append(x)
        prev = x
    return wl, frames, changed


def algorithmic(density_active_blocks, changed_pixels, macs_per_block):
    """Per-step algorithmic bytes and FLOPs of the layer step (c4 shapes)."""
    x_bytes = N_STREAMS * H * W * C * 2
    z_block_bytes = BLOCK * BLOCK * C * 4
    w_bytes = C * C * K * K * 2
    b_alg = 2 * x_bytes + changed_pixels * C * 2 + 2 * density_active_blocks * z_block_bytes + w_bytes
    flops = 2.0 * macs_per_block * density_active_blocks
    gate_bytes = 2 * x_bytes + changed_pixels * C * 2
    return b_alg, flops, gate_bytes


def flush_l2(buf):
    """Evict L2 between timed steps: write a buffer twice the L2 size, then
    read it back, so that the write-back of dirty lines (the flush's own and
    the previous step's) happens here rather than inside the next timed step.
    buf None (--no-flush): every step reads more than the L2 holds anyway."""
    if buf is None:
        return
    buf.zero_()
    buf.view(-1, 4096).amax(dim=1)


def soak(layer, frames, flush, seconds, torch):
    """Untimed steps of the same workload (with the same L2 flush between
    steps) for about `seconds`, so that the clock sampler sees the GPU under
    this load for long enough: the timed region itself lasts milliseconds."""
    t_end = time.perf_counter() + seconds
    i = 0
    while time.perf_counter() < t_end:
        for _ in range(20):
            flush_l2(flush)
            layer.step(frames[1 + i % (len(frames) - 1)])
            i += 1
        torch.cuda.synchronize()


def run_layer_timed(layer, frames, warmup, steps, flush, torch, profile=False):
    """Key frame + `warmup` untimed steps, then `steps` timed steps with an L2
    flush between them (outside the events).  Returns per-step ms, per-kernel
    (launches, ms) when profile=True, and the active-block counts."""
    from paper_2104_11487_gb300 import skipconv_profile, skipconv_profile_read
    stream = layer.stream
    layer.reset()
    t0 = time.perf_counter()
    layer.step(frames[0])
    torch.cuda.synchronize()
    key_ms = (time.perf_counter() - t0) * 1e3
    for i in range(1, warmup + 1):
        layer.step(frames[i])
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    counts = []
    skipconv_profile(layer.handle, profile)
    for i in range(steps):
        flush_l2(flush)
        ev[i][0].record(stream)
        layer.step(frames[warmup + 1 + i])
        ev[i][1].record(stream)
        if profile:
            counts.append(layer.gate()[2])
    torch.cuda.synchronize()
    launches, kms = skipconv_profile_read(layer.handle)
    ms = [a.elapsed_time(b) for a, b in ev]
    return ms, launches, kms, counts, key_ms


CONV_PATH = {"fused": 0, "separate": 3}   # AUTO (one fused launch per step) / TENSOR_CORE_SEPARATE
LAUNCH_FORMS = {0: "separate gate and convolution launches", 1: "one cooperative tensor-core launch",
                2: "one launch, a CTA per tile of gate blocks (contraction on the path named)"}


GATES = {"input": 0, "output": 2, "gumbel": 3}   # Input-Norm (mean), Output-Norm, Gumbel (Eq. 8)


def make_layer(wl, torch, dense_mode=False, path="fused", gate="input", key_interval=0):
    from paper_2104_11487_gb300 import SkipConvLayer
    phi = None
    if gate == "gumbel":
        # the gate function of Eq. 8 has no trained weights here: a seeded random one-output-channel conv
        rng = np.random.default_rng(7001)
        phi = torch.from_numpy((rng.standard_normal((1, C, K, K)) / np.sqrt(K * K * C)).astype(np.float32))
    return SkipConvLayer(N_STREAMS, C, C, H, W, k=K, stride=1, pad=1, block=BLOCK, eps=EPS, dtype="bf16",
                         dense_mode=dense_mode, conv_path=CONV_PATH[path], gate=GATES[gate],
                         key_interval=key_interval, weights=torch.from_numpy(wl.weights[0]), bias=None,
                         gate_weights=phi, gate_bias=0.0)


PROFILE_FILES = {"gate_pixel": ("gate_pixel", ("sc_gate.cu",)), "gate_block": ("gate_block", ("sc_gate.cu",)),
                 "conv": ("conv_ws", ("sc_conv_ws.cu", "sc_ws_roles.cuh", "sc_tc_common.cuh", "sc_ptx.cuh")),
                 "step_fused": ("step_fused", ("sc_step_fused.cu", "sc_ws_roles.cuh", "sc_tc_common.cuh",
                                               "sc_ptx.cuh"))}


def source_digest(files):
    import hashlib
    h = hashlib.sha256()
    for f in files:
        h.update(open(os.path.join(ROOT, "paper_2104_11487_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def traffic_from_profiles(kernel):
    """DRAM bytes per launch of `kernel` from its committed ncu summary on
    this workload, or None when there is none or the kernel's sources have
    changed since the counters were taken (the summary records the sha256 of
    the source files it was captured from)."""
    if kernel not in PROFILE_FILES:
        return None
    name, srcs = PROFILE_FILES[kernel]
    path = os.path.join(ROOT, "profiles", "%s_c4_d10.md" % name)
    if not os.path.exists(path):
        return None
    digest = source_digest(srcs)
    traffic, source_ok = None, False
    for line in open(path):
        if line.startswith("dram_bytes_per_launch:"):
            try:
                traffic = float(line.split(":", 1)[1].split()[0])
            except ValueError:
                traffic = None
        if line.startswith("source_sha256:") and line.split(":", 1)[1].strip().split()[0] == digest:
            source_ok = True
    return traffic if source_ok else None


# ----------------------------------------------------------- drift report
def drift_report(torch, intervals=(0, 4, 8, 16), T=32):
    """Skip-Conv z~ against the dense closed form z_t = w * x_t + b (a layer
    that is reset at every step) on the moving-squares workload with
    N(0, 0.01) noise (1 x 128 x 128 x 64 bf16, 8x8 blocks, eps 0.05): gates
    skip the small residuals, whose effect on z~ persists until the next key
    frame (Table 4).  Per key interval K: the largest and mean max-abs drift
    relative to RMS(z_t) over the frames, and the mean open-block density."""
    import synth
    from paper_2104_11487_gb300 import SkipConvLayer
    wl = synth.make_workload("c1", T=T)
    L = wl.layers[0]
    frames = [torch.from_numpy(np.ascontiguousarray(wl.frames[t])).cuda().to(torch.bfloat16) for t in range(T)]

    def layer(k):
        return SkipConvLayer(wl.n, L.c_in, L.c_out, wl.h, wl.w, k=L.k, stride=L.stride, pad=L.pad, block=L.block,
                             eps=L.eps, dtype="bf16", key_interval=k, weights=torch.from_numpy(wl.weights[0]),
                             bias=None if wl.biases[0] is None else torch.from_numpy(wl.biases[0]))
    ref = layer(1)
    lays = {k: layer(k) for k in intervals}
    drift = {k: [] for k in intervals}
    p99 = {k: [] for k in intervals}
    dens = {k: [] for k in intervals}
    nblk = wl.n * lays[intervals[0]].info.nby * lays[intervals[0]].info.nbx
    for x in frames:
        ref.step(x)
        zr = ref.z().double()
        rms = float(zr.pow(2).mean().sqrt())
        for k, lay in lays.items():
            lay.step(x)
            err = (lay.z().double() - zr).abs().flatten()
            drift[k].append(float(err.max()) / rms)
            p99[k].append(float(torch.kthvalue(err.cpu(), int(0.99 * err.numel())).values) / rms)
            dens[k].append(lay.gate()[2] / nblk)
    out = {}
    for k in intervals:
        d = drift[k][1:]          # frame 0 is a key frame everywhere
        out[str(k)] = {"max_rel_drift": max(d), "mean_rel_drift": sum(d) / len(d),
                       "p99_rel_drift": max(p99[k][1:]),
                       "mean_block_density": sum(dens[k][1:]) / (T - 1)}
    for lay in list(lays.values()) + [ref]:
        lay.close()
    return {"workload": "moving squares + N(0,0.01) noise, 1 x 128x128x64 bf16, 3x3, 8x8 blocks, eps 0.05, %d frames" % T,
            "reference": "the same layer reset at every step (z_t = w * x_t + b)", "key_interval": out}


# -------------------------------------------------- the other workloads
ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12      # fp32 FMA: SMs x FMA lanes x 2 FLOP x max SM clock


def layer_roof(L, n, h, w, ho, wo, esz, locs, chg, emit_y, conv_path, tc_peak, hbm):
    """Algorithmic FLOPs and bytes of one layer step and its roofline time:
    full reads of x_t and x_{t-1}, the commit of changed pixels, the fp32 z
    read-modify-write at the open locations, the weights, and y: written at
    the open locations, or (with a shortcut) refreshed over the whole frame
    from z and the shortcut.  Dense layers on the tensor path use the bf16
    tensor peak; CUDA-core layers (fp32, depthwise) the fp32 FMA peak."""
    flops = 2.0 * locs * L.c_out * (L.c_in // L.groups) * L.k * L.k
    x = n * h * w * L.c_in * esz
    bytes_ = 2 * x + chg * L.c_in * esz + 2 * locs * L.c_out * 4 + L.c_out * (L.c_in // L.groups) * L.k * L.k * esz
    if L.shortcut >= 0:
        bytes_ += n * ho * wo * L.c_out * (4 + 2 * esz)
    elif emit_y:
        bytes_ += locs * L.c_out * esz
    peak = tc_peak if conv_path == 2 else ALU_TFLOPS
    return flops, bytes_, max(flops / (peak * 1e12), bytes_ / (hbm * 1e9))


def link_stack(wl, lays):
    """Stack propagation: link each layer to the layers whose y it takes as
    x_t and as the shortcut (the frame input and external shortcuts stay
    unlinked; layers that cannot take links keep reading whole frames)."""
    from paper_2104_11487_gb300._lib import SkipConvError
    linked = 0
    for li, L in enumerate(wl.layers):
        if li == 0:
            continue
        try:
            lays[li].link(lays[li - 1], None if L.shortcut <= 0 else lays[L.shortcut - 1])
            linked += 1
        except SkipConvError:
            pass
    return linked


def workloads_report(torch, flush, tc_peak, hbm, warmup=3, names=("c0", "c1", "c2", "c3", "dw3"), link="both"):
    """The single-layer (c0, c1) and stacked (c2 pose-like, c3 MBConv-like,
    dw3 a frame-sized depthwise stack for stack propagation) workloads, run free: each layer steps on the previous layer's y (and its
    shortcut) on the device, one frame after the other, with an L2 flush
    between frames.  Frame 0 is the key frame; `warmup` frames follow
    untimed; the rest of the video is timed with CUDA events around each
    frame.  A second pass with the library's per-launch events gives each
    layer's kernel time, and a third (host-synchronised) pass counts each
    layer's open locations and changed input pixels for its roofline.
    link: "both" adds a fourth pass with the stack's layers linked (stack
    propagation, identical results); "on" links them for every pass."""
    import synth
    from paper_2104_11487_gb300 import (SkipConvLayer, device_tensor, skipconv_get_y, skipconv_profile,
                                        skipconv_profile_read)
    report = {}
    for name in names:
        wl = synth.make_workload(name)
        dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        esz = 2 if wl.dtype == "bf16" else 4
        # (a generated video may reuse one buffer for every frame: copy each frame as it comes)
        src = (wl.frames[t] for t in range(wl.T)) if isinstance(wl.frames, np.ndarray) else (f for _, f in wl.frames)
        frames = [torch.from_numpy(np.ascontiguousarray(f)).cuda().to(dt) for f in src]
        stacked = len(wl.layers) > 1
        lays, ys, dims = [], [], []
        h, w = wl.h, wl.w
        for li, L in enumerate(wl.layers):
            lay = SkipConvLayer(wl.n, L.c_in, L.c_out, h, w, k=L.k, stride=L.stride, pad=L.pad, groups=L.groups,
                                block=L.block, eps=L.eps, dtype=wl.dtype, activation=L.act, emit_y=stacked,
                                weights=torch.from_numpy(wl.weights[li]),
                                bias=None if wl.biases[li] is None else torch.from_numpy(wl.biases[li]))
            lays.append(lay)
            ys.append(device_tensor(skipconv_get_y(lay.handle), lay.shape_out, dt) if stacked else None)
            dims.append((h, w, lay.info.ho, lay.info.wo))
            h, w = lay.info.ho, lay.info.wo
        stream = lays[0].stream
        n_links = link_stack(wl, lays) if (stacked and link == "on") else 0

        def frame_step(x):
            stack = [x]
            for li, L in enumerate(wl.layers):
                lays[li].step(stack[-1], None if L.shortcut < 0 else stack[L.shortcut])
                stack.append(ys[li])

        def reset():
            for lay in lays:
                lay.reset()

        timed = range(warmup + 1, wl.T)
        # 1) whole frames
        reset()
        for t in range(warmup + 1):
            frame_step(frames[t])
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in timed]
        torch.cuda.synchronize()
        for i, t in enumerate(timed):
            flush_l2(flush)
            ev[i][0].record(stream)
            frame_step(frames[t])
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        ms = [a.elapsed_time(b) for a, b in ev]
        # 2) per-layer kernel time (library events around each launch)
        reset()
        for t in range(warmup + 1):
            frame_step(frames[t])
        for lay in lays:
            skipconv_profile(lay.handle, True)
        for t in timed:
            flush_l2(flush)
            frame_step(frames[t])
        torch.cuda.synchronize()
        layer_ms, layer_launches = [], []
        for lay in lays:
            launches, kms = skipconv_profile_read(lay.handle)
            skipconv_profile(lay.handle, False)
            layer_ms.append(sum(kms) / len(timed))
            layer_launches.append(sum(launches) / len(timed))
        # 3) open locations and changed input pixels per layer (untimed, synchronised)
        reset()
        locs = [[] for _ in lays]
        chg = [[] for _ in lays]
        prev_in = [None] * len(lays)
        for t in range(wl.T):
            stack = [frames[t]]
            for li, L in enumerate(wl.layers):
                x = stack[-1]
                if t in timed:
                    chg[li].append(int((x != prev_in[li]).any(dim=-1).sum()))
                    lays[li].step(x, None if L.shortcut < 0 else stack[L.shortcut])
                    locs[li].append(lays[li].stats()[1])
                else:
                    lays[li].step(x, None if L.shortcut < 0 else stack[L.shortcut])
                prev_in[li] = x.clone()
                stack.append(ys[li])
        per_layer, t_roof_sum, flops_sum = [], 0.0, 0.0
        for li, L in enumerate(wl.layers):
            h_, w_, ho, wo = dims[li]
            loc = statistics.mean(locs[li])
            fl, by, tr = layer_roof(L, wl.n, h_, w_, ho, wo, esz, loc, statistics.mean(chg[li]), stacked,
                                    lays[li].info.conv_path, tc_peak, hbm)
            t_roof_sum += tr
            flops_sum += fl
            per_layer.append({"layer": L.name, "shape": "%dx%dx%d -> %dx%dx%d, k%d s%d g%d, b%d" % (
                h_, w_, L.c_in, ho, wo, L.c_out, L.k, L.stride, L.groups, L.block),
                "path": {1: "cuda-core", 2: "tensor-core"}.get(lays[li].info.conv_path),
                "step_launch": LAUNCH_FORMS.get(lays[li].info.fused), "launches": layer_launches[li],
                "open_location_density": loc / (wl.n * ho * wo), "kernel_us": layer_ms[li] * 1e3,
                "eff_tflops": fl / (layer_ms[li] * 1e-3) / 1e12 if layer_ms[li] else None,
                "roofline_frac": tr / (layer_ms[li] * 1e-3) if layer_ms[li] else None})
        t_frame = statistics.median(ms) * 1e-3
        report[name] = {"frames": len(timed), "dtype": wl.dtype, "ms_per_frame": t_frame * 1e3,
                        "frames_per_s": wl.n / t_frame, "eff_tflops": flops_sum / t_frame / 1e12,
                        "stack_roofline_frac": t_roof_sum / t_frame, "layers": per_layer,
                        "linked_layers": n_links}
        if stacked and link == "both":
            # 4) the same frames with stack propagation (each layer linked to its producers)
            n_links = link_stack(wl, lays)
            reset()
            for t in range(warmup + 1):
                frame_step(frames[t])
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in timed]
            torch.cuda.synchronize()
            for i, t in enumerate(timed):
                flush_l2(flush)
                ev[i][0].record(stream)
                frame_step(frames[t])
                ev[i][1].record(stream)
            torch.cuda.synchronize()
            t_link = statistics.median([a.elapsed_time(b) for a, b in ev]) * 1e-3
            report[name]["propagation"] = {"linked_layers": n_links, "ms_per_frame": t_link * 1e3,
                                           "frames_per_s": wl.n / t_link}
        for lay in lays:
            lay.close()
        del frames
    return {"note": "frames/s and the stack roofline fraction use the median frame time (CUDA events, L2 flushed "
                    "between frames); each layer's fraction uses its kernels' event time; CUDA-core layers are "
                    "measured against %.1f TFLOP/s fp32 FMA (152 SMs x 128 lanes x 2 x 2.07 GHz)" % ALU_TFLOPS,
            "workloads": report}


# ------------------------------------------------------ warped residuals
def warped_report(torch, flush, steps=12, warmup=3):
    """Warped residuals (Eq. 10-11) under a camera pan: a 128x128x64 bf16
    texture window moving by (1, 1) px per frame, one 3x3 64->64 layer with
    8x8 blocks and eps 0.05 on the one-launch CUDA-core step.  The plain
    residual changes everywhere; warped by the pan's flow, the previous frame
    matches the current one except in the strip entering at the border.
    Per mode: median step time (CUDA events, L2 flushed between steps) and the
    mean open-block density over the timed steps."""
    import synth
    from paper_2104_11487_gb300 import SkipConvLayer
    n, h, w, c, dy, dx = 1, 128, 128, 64, 1, 1
    T = warmup + steps + 1
    v = synth.round_to_bf16(synth.panning_video(6000, T, n, h, w, c, dy, dx))
    frames = [torch.from_numpy(np.ascontiguousarray(v[t])).cuda().to(torch.bfloat16) for t in range(T)]
    wts = torch.from_numpy(synth.he_weights(np.random.default_rng(6001), c, c, 3, bf16=True))
    flow = torch.zeros((n, h, w, 2), dtype=torch.float32, device="cuda")
    flow[..., 0], flow[..., 1] = float(dy), float(dx)
    out = {"workload": "camera pan by (1, 1) px/frame over a 1 x 128x128x64 bf16 texture; 3x3 64->64, 8x8 blocks, "
                       "eps 0.05, one-launch CUDA-core step; flow = the pan", "steps": steps}
    for mode in ("plain", "warped"):
        lay = SkipConvLayer(n, c, c, h, w, k=3, block=8, eps=0.05, dtype="bf16", conv_path=1, weights=wts)
        step = (lambda x: lay.step(x)) if mode == "plain" else (lambda x: lay.step_warped(x, flow))
        for t in range(warmup + 1):
            step(frames[t])
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        torch.cuda.synchronize()
        for i in range(steps):
            flush_l2(flush)
            ev[i][0].record(lay.stream)
            step(frames[warmup + 1 + i])
            ev[i][1].record(lay.stream)
        torch.cuda.synchronize()
        us = statistics.median(a.elapsed_time(b) for a, b in ev) * 1e3
        lay.reset()
        dens = []
        for t in range(T):
            step(frames[t])
            if t > warmup:
                dens.append(lay.gate()[2] / (n * lay.info.nby * lay.info.nbx))
        out[mode] = {"us_per_step": us, "open_block_density": statistics.mean(dens)}
        lay.close()
    return out


# ----------------------------------------------------------- CPU oracle
def cpu_oracle_sample(seconds, density, max_frames=200):
    """The oracle as it stands, on the host cores: stream 0 of the same
    workload, state preset to the frame before the sample (no key frame),
    stepping frames until `seconds` of work or `max_frames`."""
    import oracle
    import synth
    wl = synth.make_workload("c4", density=density, T=max_frames + 2, n=1, h=H, w=W, c=C, block=BLOCK)
    spec = oracle.LayerSpec(n=1, c_in=C, c_out=C, h=H, w=W, k=K, block=BLOCK, eps=EPS)
    lay = oracle.OracleLayer(spec, wl.weights[0], None)
    it = iter(wl.frames)
    _, f0 = next(it)
    lay.x_prev[...] = f0
    lay.key = False
    done, t_total = 0, 0.0
    for _, f in it:
        x = np.asarray(f, np.float64)
        t0 = time.perf_counter()
        lay.step(x)
        t_total += time.perf_counter() - t0
        done += 1
        if t_total >= seconds:
            break
    return {"value": done / t_total, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
            "sample": "stream 0 of the workload, %d frames after a preset state (no key frame), %.1f s, "
                      "double-precision C loops" % (done, t_total)}


def cpu_model() -> str:
    """The host CPU's model name (lscpu / /proc/cpuinfo), else the machine type."""
    import platform
    import subprocess
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.machine()


def cpu_workload_sample(name, seconds, threads):
    """The oracle stepping a whole workload (every layer of a stack) on the
    host cores: the key frame untimed on all cores, then frames 1, 2, ... timed
    with `threads` threads until `seconds` of work (at least one frame) or the
    end of the video."""
    import oracle
    import synth
    wl = synth.make_workload(name)
    refs, shortcuts = [], []
    h, w = wl.h, wl.w
    for li, L in enumerate(wl.layers):
        spec = oracle.LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=h, w=w, k=L.k, stride=L.stride, pad=L.pad,
                                groups=L.groups, block=L.block, eps=L.eps)
        refs.append(oracle.OracleLayer(spec, wl.weights[li], wl.biases[li]))
        h, w = spec.ho, spec.wo
    round_mode = 2 if wl.dtype == "bf16" else 1

    def frame(x):
        stack = [np.asarray(x, np.float64)]
        for li, L in enumerate(wl.layers):
            refs[li].step(stack[-1])
            if len(wl.layers) > 1:
                sc = None if L.shortcut < 0 else stack[L.shortcut]
                stack.append(oracle.layer_output(refs[li].z, sc, L.act, round_mode))

    cores = oracle.num_threads()
    frame(wl.frames[0])
    oracle.set_num_threads(threads)
    done, t_total = 0, 0.0
    try:
        for t in range(1, wl.T):
            t0 = time.perf_counter()
            frame(wl.frames[t])
            t_total += time.perf_counter() - t0
            done += 1
            if t_total >= seconds:
                break
    finally:
        oracle.set_num_threads(cores)
    return {"frames_per_s": wl.n * done / t_total, "ms_per_frame": t_total / done * 1e3, "threads": threads,
            "sample": "frames 1-%d after the key frame (%d layers)" % (done, len(wl.layers))}


def cpu_baseline_table(seconds_each):
    """The oracle on every workload, at all host cores and at one: c0-c3 as
    whole stacks (frames/s) and the c4 layer at each sweep density (stream 0,
    stream-frames/s).  One core takes c4 only up to 10 % density: a single
    frame at 50 % is about 10 GFLOP of double-precision loops."""
    import oracle
    cores = oracle.num_threads()
    rows = []
    for name in ("c0", "c1", "c2", "c3"):
        for threads in (cores, 1):
            r = cpu_workload_sample(name, seconds_each, threads)
            r["workload"] = name
            rows.append(r)
    from synth.workloads import C4_DENSITIES
    for d in C4_DENSITIES:
        for threads in (cores, 1):
            if threads == 1 and d > 0.10:
                continue
            oracle.set_num_threads(threads)
            try:
                r = cpu_oracle_sample(seconds_each, d, max_frames=60)
            finally:
                oracle.set_num_threads(cores)
            rows.append({"workload": "c4 d=%g" % d, "frames_per_s": r["value"], "ms_per_frame": 1e3 / r["value"],
                         "threads": threads, "sample": r["sample"]})
    return {"cpu": cpu_model(), "cores": cores, "seconds_per_sample": seconds_each,
            "unit": "frames/s (c4: stream-frames/s of stream 0)", "rows": rows}


# ------------------------------------------------------------- ranks
class Ranks:
    """Process-group plumbing of a replica run (torchrun, one rank per GPU):
    every rank runs its own streams, there is no collective on the data path;
    ranks meet only at barriers around the timed region and to take the
    slowest rank's time.  backend/device: "nccl"/"cuda" on GPUs, "gloo"/"cpu"
    in the CPU tests."""

    def __init__(self, backend="nccl", device="cuda"):
        import torch
        self.torch = torch
        self.rank = int(os.environ.get("RANK", "0"))
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.device = device
        self.dist = None
        if self.world > 1:
            import torch.distributed as dist
            kw = {"device_id": torch.device("cuda", self.local)} if device == "cuda" else {}
            dist.init_process_group(backend, **kw)
            self.dist = dist

    def barrier(self):
        if self.dist:
            self.dist.barrier()
        if self.device == "cuda":
            self.torch.cuda.synchronize()

    def max(self, v: float) -> float:
        """The largest v over all ranks (the slowest rank's time)."""
        if not self.dist:
            return v
        t = self.torch.tensor([v], dtype=self.torch.float64, device=self.device)
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.dist:
            self.dist.destroy_process_group()


def replica_value(world: int, steps: int, total_ms: float) -> float:
    """Whole-job stream-frames/s: the stream-frames of all ranks over the
    slowest rank's time."""
    return world * N_STREAMS * steps / (total_ms / 1e3)


# ---------------------------------------------------------------- main
def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return 0
        return run_reference(args)

    import torch
    torch.cuda.set_device(local)
    ranks = Ranks()
    barrier, max_over_ranks = ranks.barrier, ranks.max

    from paper_2104_11487_gb300 import _lib, skipconv_get_info
    _lib.lib()
    pk, pk_src = peaks()
    hbm, tc_peak = pk["hbm_gbs"], pk["bf16_tflops"]

    if args.workloads_only:
        flush = None if args.no_flush else torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
        names = [x for x in args.workloads_only.split(",") if x]
        out = {}
        if "warped" in names:
            names.remove("warped")
            out["warped_residual"] = warped_report(torch, flush)
        if names:
            out["other_workloads"] = workloads_report(torch, flush, tc_peak, hbm, names=tuple(names), link=args.link)
        if rank == 0:
            print(json.dumps(out), flush=True)
        ranks.close()
        return 0

    n_frames = args.warmup + args.steps + 1
    wl, frames, changed = device_frames(args.density, n_frames, rank, torch)
    flush = None if args.no_flush else torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    layer = make_layer(wl, torch, path=args.path, gate=args.gate, key_interval=args.key_interval)
    info = skipconv_get_info(layer.handle)

    # 1) headline: timed steps, no per-kernel events
    clocks = Clocks(local, args.clocks_log)
    barrier()
    clocks.start()
    if not args.no_soak:
        soak(layer, frames, flush, 0.5, torch)
    barrier()
    ms, launches, _, _, key_ms = run_layer_timed(layer, frames, args.warmup, args.steps, flush, torch)
    barrier()
    if not args.no_soak:
        soak(layer, frames, flush, 0.5, torch)
    clk = clocks.stop()
    clk["window"] = "every 100 ms over the timed steps and 0.5 s of the same steps before and after"
    total_ms = max_over_ranks(sum(ms))
    ms_per_step = total_ms / args.steps
    value = replica_value(world, args.steps, total_ms)

    # 2) the same steps with per-kernel CUDA events (dominant kernel's roofline)
    ms_p, launches_p, kms, counts, _ = run_layer_timed(layer, frames, args.warmup, args.steps, flush, torch,
                                                       profile=True)
    active = statistics.mean(counts) if counts else 0.0
    chg = statistics.mean(changed[args.warmup:args.warmup + args.steps]) if changed else 0.0
    macs_per_block = BLOCK * BLOCK * C * C * K * K
    b_alg, flops, gate_bytes = algorithmic(active, chg, macs_per_block)
    t_step = ms_per_step / 1e3
    t_roof = max(flops / (tc_peak * 1e12), b_alg / (hbm * 1e9))
    per_kernel = {KERNELS[k]: {"launches": launches_p[k], "avg_us": (kms[k] / launches_p[k] * 1e3)
                               if launches_p[k] else None} for k in range(len(KERNELS))}
    dom = max((0, 1, 2, 4), key=lambda k: kms[k])
    dom_us = kms[dom] / max(1, launches_p[dom]) * 1e3
    if dom == 4:
        # the fused kernel is the whole step: its algorithmic bytes are the step's
        bound_tc = flops / (tc_peak * 1e12) > b_alg / (hbm * 1e9)
        if bound_tc:
            ach = flops / (dom_us * 1e-6) / 1e12
            roof = {"kernel": "step_fused", "bound": "tensor", "achieved": ach, "peak": tc_peak, "unit": "TFLOP/s",
                    "frac": ach / tc_peak, "peak_source": pk_src + " bf16_tflops (burst)",
                    "traffic": traffic_from_profiles("step_fused")}
        else:
            ach = b_alg / (dom_us * 1e-6) / 1e9
            roof = {"kernel": "step_fused", "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                    "frac": ach / hbm, "peak_source": pk_src + " hbm_gbs", "algorithmic_bytes_per_launch": b_alg,
                    "traffic": traffic_from_profiles("step_fused")}
    elif dom == 2:
        ach = flops / (dom_us * 1e-6) / 1e12
        roof = {"kernel": "conv", "bound": "tensor", "achieved": ach, "peak": tc_peak, "unit": "TFLOP/s",
                "frac": ach / tc_peak, "peak_source": pk_src + " bf16_tflops (burst)",
                "traffic": traffic_from_profiles("conv")}
    else:
        ach = gate_bytes / (dom_us * 1e-6) / 1e9 if dom == 0 else None
        # the Gumbel gate's passes are other kernels than the ones the committed summaries profile
        name = KERNELS[dom] + ("_gumbel" if args.gate == "gumbel" else "")
        roof = {"kernel": name, "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                "frac": (ach / hbm) if ach else None, "peak_source": pk_src + " hbm_gbs",
                "algorithmic_bytes_per_launch": gate_bytes,
                "traffic": None if args.gate == "gumbel" else traffic_from_profiles(KERNELS[dom])}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded block-perturbation video)",
            "config": workload_config(args.density, flushed=not args.no_flush, gate=args.gate,
                                      key_interval=args.key_interval),
            "conv_path": {1: "cuda-core", 2: "tensor-core"}.get(info.conv_path),
            "step_launches": LAUNCH_FORMS.get(info.fused),
            "active_blocks_per_step": active, "block_density_measured": active / (N_STREAMS * (H // BLOCK) ** 2),
            "changed_pixels_per_step": chg,
            "eff_tflops": flops / t_step / 1e12,
            "step_roofline": {"t_roof_us": t_roof * 1e6, "t_meas_us": t_step * 1e6, "frac": t_roof / t_step,
                              "bytes_alg": b_alg, "flops_active": flops, "peaks": pk_src},
            "key_frame_ms_host": key_ms,
            "per_kernel": per_kernel, "roofline": roof,
            "gpu_launches": int(sum(launches)), "clocks": clk}

    # 3) end to end through the host-buffer ABI call (pinned host frames, z read back)
    if not args.no_e2e:
        from paper_2104_11487_gb300 import skipconv_step_host, skipconv_step_host_async, skipconv_sync
        host = [f.cpu().pin_memory() for f in frames]
        zh = [torch.empty((N_STREAMS, H, W, C), dtype=torch.float32).pin_memory() for _ in range(2)]
        # one untimed round trip through every pinned buffer first: the first copies out of freshly pinned
        # host memory were measured at 3-5 ms per 192 MiB step against 1.07 ms once the buffers had been
        # used, and a caller allocates its pinned buffers once
        scratch = torch.empty_like(frames[0])
        for hb in host:
            scratch.copy_(hb, non_blocking=True)
        zscratch = torch.empty((N_STREAMS, H, W, C), dtype=torch.float32, device="cuda")
        for zb in zh:
            zb.copy_(zscratch, non_blocking=True)
        torch.cuda.synchronize()
        del scratch, zscratch
        # synchronous calls: each step uploads, steps, downloads and waits
        layer.reset()
        for i in range(args.warmup + 1):
            skipconv_step_host(layer.handle, host[i], zh[0])
        barrier()
        t0 = time.perf_counter()
        for i in range(args.steps):
            skipconv_step_host(layer.handle, host[args.warmup + 1 + i], zh[0])
        t_sync = max_over_ranks(time.perf_counter() - t0)
        # pipelined calls: the upload of step t+1 and the download of step t-1 overlap step t; the timed
        # region ends when the last step's z is in host memory
        layer.reset()
        for i in range(args.warmup + 1):
            skipconv_step_host_async(layer.handle, host[i], zh[i % 2])
        skipconv_sync(layer.handle)
        barrier()
        t0 = time.perf_counter()
        for i in range(args.steps):
            skipconv_step_host_async(layer.handle, host[args.warmup + 1 + i], zh[i % 2])
        skipconv_sync(layer.handle)
        t_e2e = max_over_ranks(time.perf_counter() - t0)
        # the sparse result: each step's open blocks of z (count, ids, values) written by the device straight
        # into pinned host memory -- what a consumer holding z needs (Eq. 3 changes z only there)
        from paper_2104_11487_gb300 import skipconv_step_host_sparse_async
        nblk = N_STREAMS * (H // BLOCK) * (W // BLOCK)
        zbk = [torch.empty((nblk, BLOCK, BLOCK, C), dtype=torch.float32).pin_memory() for _ in range(2)]
        lbk = [torch.empty(nblk, dtype=torch.int32).pin_memory() for _ in range(2)]
        cbk = [torch.zeros(1, dtype=torch.int32).pin_memory() for _ in range(2)]
        layer.reset()
        for i in range(args.warmup + 1):
            skipconv_step_host_sparse_async(layer.handle, host[i], zbk[i % 2], lbk[i % 2], cbk[i % 2])
        skipconv_sync(layer.handle)
        barrier()
        t0 = time.perf_counter()
        for i in range(args.steps):
            skipconv_step_host_sparse_async(layer.handle, host[args.warmup + 1 + i], zbk[i % 2], lbk[i % 2],
                                            cbk[i % 2])
        skipconv_sync(layer.handle)
        t_sparse = max_over_ranks(time.perf_counter() - t0)
        # bytes the result took over the link: an untimed pass reading each step's count
        layer.reset()
        for i in range(args.warmup + 1):
            skipconv_step_host_sparse_async(layer.handle, host[i], zbk[0], lbk[0], cbk[0])
        skipconv_sync(layer.handle)
        cnts = []
        for i in range(args.steps):
            skipconv_step_host_sparse_async(layer.handle, host[args.warmup + 1 + i], zbk[0], lbk[0], cbk[0])
            skipconv_sync(layer.handle)
            cnts.append(int(cbk[0][0]))
        d2h_sparse = 4 + statistics.mean(cnts) * (4 + BLOCK * BLOCK * C * 4)
        line["e2e"] = {"value": replica_value(world, args.steps, t_sparse * 1e3), "unit": UNIT,
                       "h2d_bytes_per_step": host[0].numel() * 2, "d2h_bytes_per_step": d2h_sparse,
                       "call": "skipconv_step_host_sparse_async then skipconv_sync (host frame in; the step's open "
                               "blocks of fp32 z, their ids and count out, written by the device into pinned "
                               "host memory; uploads of neighbouring steps overlap)",
                       "full_z_value": replica_value(world, args.steps, t_e2e * 1e3),
                       "full_z_d2h_bytes_per_step": zh[0].numel() * 4,
                       "full_z_call": "skipconv_step_host_async then skipconv_sync (host frame in, full fp32 z out; "
                                      "copies of neighbouring steps overlap)",
                       "sync_value": replica_value(world, args.steps, t_sync * 1e3),
                       "sync_call": "skipconv_step_host (one synchronous call per step, full z out)"}
        del host, zbk

    # 4) density sweep vs the all-ones dense mode of the same kernels
    if not args.no_sweep:
        sweep = []
        del frames
        dense_ms = None
        for d in (0.0, 0.01, 0.05, 0.10, 0.25, 0.50, 1.00):
            wl_d, fr_d, ch_d = device_frames(d, args.warmup + args.sweep_steps + 1, rank, torch)
            lay_d = make_layer(wl_d, torch, path=args.path, gate=args.gate, key_interval=args.key_interval)
            # timed as the headline is (no per-launch events, no read-back between steps), then an untimed
            # pass of the same steps for the open-block counts
            ms_d, *_ = run_layer_timed(lay_d, fr_d, args.warmup, args.sweep_steps, flush, torch)
            _, _, _, cnt_d, _ = run_layer_timed(lay_d, fr_d, args.warmup, args.sweep_steps, flush, torch,
                                                profile=True)
            if d == 0.10:
                lay_dense = make_layer(wl_d, torch, dense_mode=True, path=args.path, gate=args.gate)
                ms_dn, _, _, _, _ = run_layer_timed(lay_dense, fr_d, args.warmup, args.sweep_steps, flush, torch)
                dense_ms = statistics.median(ms_dn)
                lay_dense.close()
            act = statistics.mean(cnt_d)
            chg_d = statistics.mean(ch_d[args.warmup:]) if ch_d else 0.0
            b_d, f_d, _ = algorithmic(act, chg_d, macs_per_block)
            t_d = statistics.median(ms_d) / 1e3
            sweep.append({"density": d, "active_blocks": act, "ms_per_step": t_d * 1e3,
                          "frames_per_s": N_STREAMS / t_d, "eff_tflops": f_d / t_d / 1e12,
                          "step_roofline_frac": max(f_d / (tc_peak * 1e12), b_d / (hbm * 1e9)) / t_d})
            lay_d.close()
            del fr_d
        for s in sweep:
            s["faster_than_dense_mode"] = (s["ms_per_step"] < dense_ms) if dense_ms else None
        line["sweep"] = {"points": sweep, "dense_mode_ms_per_step": dense_ms}

    # 5) the single-layer and stacked workloads
    if not args.no_workloads:
        line["other_workloads"] = workloads_report(torch, flush, tc_peak, hbm, link=args.link)

    if not args.no_workloads:
        line["warped_residual"] = warped_report(torch, flush)

    # 6) the CPU oracle on the host cores (rank 0, N = 1 only)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_oracle_sample(args.cpu_seconds, args.density)
        # the same oracle on one host core (a shorter sample)
        import oracle
        cores = oracle.num_threads()
        oracle.set_num_threads(1)
        one = cpu_oracle_sample(args.cpu_seconds / 3, args.density)
        oracle.set_num_threads(cores)
        line["cpu_baseline"]["single_core"] = {"value": one["value"], "unit": one["unit"], "sample": one["sample"]}
        if not args.no_cpu_table:
            line["cpu_baseline"]["per_workload"] = cpu_baseline_table(args.cpu_table_seconds)
    layer.close()
    if args.drift and rank == 0:
        line["drift_vs_dense"] = drift_report(torch)
    if rank == 0:
        print(json.dumps(line), flush=True)
    ranks.close()
    return 0


def run_reference(args):
    """The oracle arm: each step is the oracle on a bounded sample of the
    workload (stream 0, one frame), on the host cores."""
    import oracle
    import synth
    n_frames = args.warmup + args.steps + 1
    wl = synth.make_workload("c4", density=args.density, T=n_frames + 1, n=1, h=H, w=W, c=C, block=BLOCK)
    spec = oracle.LayerSpec(n=1, c_in=C, c_out=C, h=H, w=W, k=K, block=BLOCK, eps=EPS)
    lay = oracle.OracleLayer(spec, wl.weights[0], None)
    it = iter(wl.frames)
    _, f0 = next(it)
    lay.x_prev[...] = f0
    lay.key = False
    times = []
    for i, (_, f) in enumerate(it):
        x = np.asarray(f, np.float64)
        t0 = time.perf_counter()
        lay.step(x)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.append(dt)
        if len(times) >= args.steps:
            break
    total = sum(times)
    value = len(times) / total
    sample = "oracle (double-precision C loops) on stream 0 of the workload, one frame per step, state preset"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1,
            "steps": len(times), "warmup": args.warmup, "ms_per_step": total / len(times) * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded block-perturbation video)", "config": workload_config(args.density),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
