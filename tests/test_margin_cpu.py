"""The generators' eps-margin record (synth.workloads.MARGIN_REDRAWS), checked
with the oracle on the CPU.

Every gate decision of a parity input should be decided by more than rounding:
no block score within 2e-5 (relative) of eps, twice the parity tests' band.
For each workload at its stated size, the recorded redraw index must be the
first whose frames keep that margin: every lower index has at least one
decision inside it, the recorded one none.  The parity tests then assert that
no block is excluded.
"""
import numpy as np
import pytest

import margin
import synth
from oracle import LayerSpec
from synth.workloads import MARGIN_REDRAWS


def events(name, redraw, **kw):
    wl = synth.make_workload(name, redraw=redraw, **kw)
    if len(wl.layers) > 1:
        return sum(margin.stack_band_events(wl))
    L = wl.layers[0]
    spec = LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=wl.h, w=wl.w, k=L.k, stride=L.stride, pad=L.pad,
                     groups=L.groups, block=L.block, eps=L.eps)
    frames = wl.frames if isinstance(wl.frames, np.ndarray) else [f.copy() for _, f in wl.frames]
    return margin.layer_band_events(spec, frames, wl.weights[0])


@pytest.mark.parametrize("name", ["c0", "c1", "c2", "c3"])
def test_recorded_redraw_is_the_first_with_the_margin(name):
    r = MARGIN_REDRAWS[name]
    assert events(name, r) == 0, "%s: redraw %d has gate decisions within the margin" % (name, r)
    for lower in range(r):
        assert events(name, lower) > 0, "%s: redraw %d already keeps the margin" % (name, lower)


def test_block_perturbation_video_keeps_the_margin():
    """The density sweep's frames change only inside the perturbed blocks
    (their 6x6 interior), so every other block's score is exactly 0 and every
    perturbed block's is far above eps: checked at the bench's 10 % density on
    two streams of the full frame size and channel count."""
    assert MARGIN_REDRAWS["c4"] == 0
    assert events("c4", 0, density=0.10, T=8, n=2) == 0


def test_margin_band_catches_a_near_eps_score():
    """The margin test itself: a residual built so that one block's mean score
    lies 1e-5 (relative) above eps is counted; at 3e-5 it is not."""
    spec = LayerSpec(n=1, c_in=4, c_out=4, h=8, w=8, k=3, block=4, eps=0.05)
    for rel, expect in ((1e-5, 1), (3e-5, 0)):
        x0 = np.zeros((1, 8, 8, 4))
        x1 = x0.copy()
        # one changed pixel at the centre of block (0, 0): the largest support mean is |d| / (4 * 9)
        x1[0, 1, 1, :] = spec.eps * (1 + rel) * 9.0
        assert margin.layer_band_events(spec, [x0, x1]) == expect
