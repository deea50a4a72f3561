"""The five Skip-Conv workloads: layer shapes, stacks and seeded inputs.

c0  single 3x3 layer, 32->32 channels, 64x64, T=8, fp32, 1x1 gate blocks, eps 0.05
c1  single 3x3 layer, 64->64, 128x128, T=16, bf16, 8x8 blocks, eps 0.05
c2  HRNet-W32-like pose stack on 256x192, T=32, bf16, 4x4 blocks, eps 0.05
c3  EfficientDet-D0-like MBConv stack at 64x64x40 (1/8 of 512x512), T=32, bf16,
    8x8 blocks, eps 0.03
c4  single 3x3 layer, 256->256, 8 streams of 128x128, T=32, bf16, 8x8 blocks,
    eps 0.05, with a per-frame changed-block density d

Seeds are 1000*config + stream.  Every dimension can be scaled down through
keyword overrides for the small parity cases.

Redraws.  A gate decision whose score lies within a hair of eps is decided by
rounding, so the parity tests need inputs that keep every gate score away from
eps.  ``redraw=r`` draws the frames from seed base + REDRAW_STRIDE * r instead
of the base seed (weights keep their seed); ``MARGIN_REDRAWS`` records, per
workload at its stated size, the first redraw index whose inputs keep the
margin (a CPU test recomputes it with the oracle).  This module only draws: it
does not compute gate scores.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from .video import (block_perturbation_video, he_weights, moving_rect_video,
                    moving_squares_video, round_to_bf16, traffic_video)

ACT_NONE, ACT_RELU, ACT_SILU = 0, 1, 2

REDRAW_STRIDE = 100000
# First redraw index whose frames keep every gate score at least 2e-5 (relative)
# away from eps, for each workload at its stated size (the margin test in
# tests/ recomputes these with the oracle and checks that every lower index fails).
MARGIN_REDRAWS = {"c0": 0, "c1": 0, "c2": 1, "c3": 0, "c4": 0}


def _seed(base: int, redraw: int) -> int:
    return base + REDRAW_STRIDE * int(redraw)


@dataclass
class LayerDef:
    """One Skip-Conv layer of a workload.  `shortcut` names the index of the
    stack tensor added before the activation (-1: none; 0 is the stack input,
    l+1 the output of layer l)."""
    c_in: int
    c_out: int
    k: int
    stride: int
    pad: int
    groups: int
    block: int
    eps: float
    act: int = ACT_NONE
    shortcut: int = -1
    name: str = ""


@dataclass
class Workload:
    name: str
    dtype: str                      # "f32" or "bf16" (frames, weights, layer outputs)
    n: int                          # independent streams
    h: int
    w: int
    c: int
    T: int
    layers: list
    weights: list = field(default_factory=list)   # float32 arrays, [c_out][c_in/g][k][k]
    biases: list = field(default_factory=list)    # float32 arrays or None
    frames: object = None           # float32 [T, n, h, w, c] or an iterable of (t, frame)


def _weights(seed: int, layers, bf16: bool, bias_std: float):
    rng = np.random.default_rng(seed)
    ws, bs = [], []
    for L in layers:
        ws.append(he_weights(rng, L.c_out, L.c_in // L.groups, L.k, bf16))
        if bias_std > 0:
            b = (rng.standard_normal(L.c_out) * bias_std).astype(np.float32)
            bs.append(round_to_bf16(b) if bf16 else b)
        else:
            bs.append(None)
    return ws, bs


def c0(T: int = 8, h: int = 64, w: int = 64, c: int = 32, redraw: int = 0) -> Workload:
    layers = [LayerDef(c, c, 3, 1, 1, 1, 1, 0.05, name="conv3x3")]
    frames = moving_squares_video(_seed(0, redraw), T, h, w, c, n_squares=3, size=8, speed=2, noise_std=0.01)
    ws, bs = _weights(1, layers, bf16=False, bias_std=0.0)
    return Workload("c0", "f32", 1, h, w, c, T, layers, ws, bs, frames[:, None])


def c1(T: int = 16, h: int = 128, w: int = 128, c: int = 64, n_squares: int = 6, size: int = 16,
       redraw: int = 0) -> Workload:
    layers = [LayerDef(c, c, 3, 1, 1, 1, 8, 0.05, name="conv3x3")]
    frames = round_to_bf16(moving_squares_video(_seed(1000, redraw), T, h, w, c, n_squares=n_squares, size=size,
                                                speed=2, noise_std=0.01))
    ws, bs = _weights(1001, layers, bf16=True, bias_std=0.0)
    return Workload("c1", "bf16", 1, h, w, c, T, layers, ws, bs, frames[:, None])


def c2_layers(block: int = 4, eps: float = 0.05, width: int = 32, stem: int = 64, n_blocks: int = 4):
    L = [LayerDef(3, stem, 3, 2, 1, 1, block, eps, ACT_RELU, name="stem1"),
         LayerDef(stem, stem, 3, 2, 1, 1, block, eps, ACT_RELU, name="stem2"),
         LayerDef(stem, width, 3, 1, 1, 1, block, eps, ACT_RELU, name="transition")]
    for bi in range(n_blocks):
        inp = len(L)                        # stack index of this basic block's input
        L.append(LayerDef(width, width, 3, 1, 1, 1, block, eps, ACT_RELU, name=f"block{bi}.conv1"))
        L.append(LayerDef(width, width, 3, 1, 1, 1, block, eps, ACT_RELU, shortcut=inp,
                          name=f"block{bi}.conv2"))
    return L


def c2(T: int = 32, h: int = 256, w: int = 192, n_blocks: int = 4, redraw: int = 0) -> Workload:
    layers = c2_layers(n_blocks=n_blocks)
    frames = round_to_bf16(moving_rect_video(_seed(2000, redraw), T, h, w, 3, n_rects=2, rh=48, rw=32, speed=2, jitter=1))
    ws, bs = _weights(2001, layers, bf16=True, bias_std=0.01)
    return Workload("c2", "bf16", 1, h, w, 3, T, layers, ws, bs, frames[:, None])


def c3_layers(block: int = 8, eps: float = 0.03, c: int = 40, expand: int = 240, n_blocks: int = 3):
    L = []
    for bi in range(n_blocks):
        inp = len(L)
        L.append(LayerDef(c, expand, 1, 1, 0, 1, block, eps, ACT_SILU, name=f"mb{bi}.expand"))
        L.append(LayerDef(expand, expand, 3, 1, 1, expand, block, eps, ACT_SILU, name=f"mb{bi}.dw"))
        L.append(LayerDef(expand, c, 1, 1, 0, 1, block, eps, ACT_NONE, shortcut=inp, name=f"mb{bi}.project"))
    return L


def c3(T: int = 32, n_blocks: int = 3, redraw: int = 0) -> Workload:
    """512x512x3 traffic-like video, 8x8 average-pooled to 64x64x3 and lifted
    to 40 channels by a fixed seeded 1x1 map (input preparation, untimed)."""
    raw = traffic_video(_seed(3000, redraw), T)
    pooled = raw.reshape(T, 64, 8, 64, 8, 3).mean(axis=(2, 4), dtype=np.float64).astype(np.float32)
    rng = np.random.default_rng(3002)
    lift = (rng.standard_normal((3, 40)) / np.sqrt(3.0)).astype(np.float32)
    frames = round_to_bf16(np.einsum("thwc,cd->thwd", pooled, lift).astype(np.float32))
    layers = c3_layers(n_blocks=n_blocks)
    ws, bs = _weights(3001, layers, bf16=True, bias_std=0.01)
    return Workload("c3", "bf16", 1, 64, 64, 40, T, layers, ws, bs, frames[:, None])


C4_DENSITIES = (0.0, 0.01, 0.05, 0.10, 0.25, 0.50, 1.00)


def c4(density: float = 0.10, T: int = 32, n: int = 8, h: int = 128, w: int = 128, c: int = 256,
       block: int = 8, dtype: str = "bf16", stream_offset: int = 0, redraw: int = 0) -> Workload:
    """Density sweep layer.  `frames` is an iterable yielding (t, frame);
    `stream_offset` selects other streams' seeds (independent replicas)."""
    layers = [LayerDef(c, c, 3, 1, 1, 1, block, 0.05, name="conv3x3")]
    n_changed = int(round(density * (h // block) * (w // block)))
    bf16 = dtype == "bf16"
    frames = block_perturbation_video(_seed(4000, redraw), T, n, h, w, c, block, n_changed, bf16=bf16,
                                      stream_offset=stream_offset)
    ws, bs = _weights(4001, layers, bf16=bf16, bias_std=0.0)
    return Workload("c4", dtype, n, h, w, c, T, layers, ws, bs, frames)


def dw3(density: float = 0.10, T: int = 16, n: int = 8, h: int = 128, w: int = 128, c: int = 128,
        block: int = 8) -> Workload:
    """A frame-sized stack for stack propagation: three depthwise 3x3 layers
    (c channels, ReLU between) on c4's block-perturbation video -- each layer
    streams two 32 MiB frames per step in full, while only the perturbed blocks
    and their halo change.  `frames` is an iterable yielding (t, frame)."""
    layers = [LayerDef(c, c, 3, 1, 1, c, block, 0.05, ACT_RELU, name="dw%d" % i) for i in range(3)]
    n_changed = int(round(density * (h // block) * (w // block)))
    frames = block_perturbation_video(5000, T, n, h, w, c, block, n_changed, bf16=True)
    ws, bs = _weights(5001, layers, bf16=True, bias_std=0.01)
    return Workload("dw3", "bf16", n, h, w, c, T, layers, ws, bs, frames)


WORKLOADS = {"c0": c0, "c1": c1, "c2": c2, "c3": c3, "c4": c4, "dw3": dw3}


def make_workload(name: str, **kw) -> Workload:
    """The named workload.  Without an explicit ``redraw``, the workloads that
    record one in MARGIN_REDRAWS use it."""
    if "redraw" not in kw and name in MARGIN_REDRAWS:
        kw["redraw"] = MARGIN_REDRAWS[name]
    return WORKLOADS[name](**kw)
