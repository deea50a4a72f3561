"""Free-running stacks against the oracle's free-running stacks (c2 pose-like,
c3 MBConv-like): each side feeds every layer its own previous layer's
y = round(act(z [+ shortcut])).  Stack parity proper is teacher-forced
(test_parity_gpu): here a one-ulp bf16 difference upstream may flip a gate
near eps, and under the literal x_{t-1} reading that flip persists, so this
run is reported, not held bit-exact.  What must hold: the key frame opens
every block on both sides and its output matches within a few rounding
steps of the bf16 chain; afterwards the gate masks agree on nearly every
block of every layer and the output stays close to the oracle's."""
import numpy as np
import pytest
import torch

import synth
from harness import gpu_layer, to_device
from oracle import LayerSpec, OracleLayer, layer_output

pytestmark = pytest.mark.gpu


def run_free(wl, frames):
    h, w = wl.h, wl.w
    refs, gls = [], []
    for li, L in enumerate(wl.layers):
        spec = LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=h, w=w, k=L.k, stride=L.stride, pad=L.pad,
                         groups=L.groups, block=L.block, eps=L.eps)
        refs.append((spec, OracleLayer(spec, wl.weights[li], wl.biases[li])))
        gls.append(gpu_layer(spec, wl.weights[li], wl.biases[li], wl.dtype, act=L.act, emit_y=True))
        h, w = spec.ho, spec.wo
    round_mode = 2 if wl.dtype == "bf16" else 1
    agree = np.zeros((len(frames), len(wl.layers)))
    out_err = []
    try:
        for t, frame in enumerate(frames):
            ref_stack = [np.asarray(frame, np.float64)]
            gpu_stack = [to_device(frame, wl.dtype)]
            for li, L in enumerate(wl.layers):
                spec, ref = refs[li]
                _, mask_ref = ref.step(ref_stack[-1])
                sc_ref = None if L.shortcut < 0 else ref_stack[L.shortcut]
                ref_stack.append(layer_output(ref.z, sc_ref, L.act, round_mode))
                gls[li].step(gpu_stack[-1], None if L.shortcut < 0 else gpu_stack[L.shortcut])
                mask = gls[li].gate()[0].cpu().numpy()
                agree[t, li] = float(np.mean(mask.astype(bool) == mask_ref.astype(bool)))
                if t == 0:
                    assert mask.all() and mask_ref.all(), "%s layer %s: the key frame must open every block" % (
                        wl.name, L.name)
                gpu_stack.append(gls[li].y())
            y_ref = ref_stack[-1]
            y_gpu = gpu_stack[-1].float().cpu().numpy().astype(np.float64)
            rms = float(np.sqrt(np.mean(y_ref ** 2)))
            out_err.append((float(np.abs(y_gpu - y_ref).max()) / rms, float(np.sqrt(np.mean((y_gpu - y_ref) ** 2))) / rms))
    finally:
        for g in gls:
            g.close()
    return agree, out_err


@pytest.mark.parametrize("name", ["c2", "c3"])
def test_free_running_stack_tracks_the_oracle(name):
    wl = synth.make_workload(name)
    agree, err = run_free(wl, [wl.frames[t] for t in range(12)])
    print("\n%s free-running, 12 frames: mask agreement per layer (min over frames): %s" % (
        name, " ".join("%.4f" % v for v in agree.min(axis=0))))
    print("%s last layer y: max-abs / RMS per frame %s; RMS error / RMS %s" % (
        name, " ".join("%.3g" % e[0] for e in err), " ".join("%.2g" % e[1] for e in err)))
    # the key frame: every gate open, only rounding in the chain
    assert err[0][1] < 1e-2, err[0]
    # afterwards: flips near eps persist, but they stay rare and local
    assert agree.mean(axis=0).min() >= 0.97, agree.mean(axis=0)
    assert max(e[1] for e in err) < 5e-2, err
