"""Stack propagation (skipconv_link_inputs): a linked layer skips the tiles
whose inputs did not change, and must produce exactly what the unlinked
layer produces -- z, y, gate masks, open-block lists and the committed
x_{t-1}, bit for bit, at every layer and frame of the c2 (pose-like) and c3
(MBConv-like) stacks run free (each layer on the previous layer's y on the
device), including key frames in the middle and a producer that steps twice
between two steps of its consumer."""
import numpy as np
import pytest
import torch

import synth
from paper_2104_11487_gb300 import SkipConvLayer, device_tensor, skipconv_get_y
from paper_2104_11487_gb300._lib import SKIPCONV_ERR_INVALID, SKIPCONV_ERR_UNSUPPORTED, SkipConvError

pytestmark = pytest.mark.gpu


def build_stack(wl, link, key_interval=None):
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    lays, ys = [], []
    h, w = wl.h, wl.w
    for li, L in enumerate(wl.layers):
        ki = 0 if key_interval is None else key_interval.get(li, 0)
        lay = SkipConvLayer(wl.n, L.c_in, L.c_out, h, w, k=L.k, stride=L.stride, pad=L.pad, groups=L.groups,
                            block=L.block, eps=L.eps, dtype=wl.dtype, activation=L.act, emit_y=True,
                            weights=torch.from_numpy(wl.weights[li]), key_interval=ki,
                            bias=None if wl.biases[li] is None else torch.from_numpy(wl.biases[li]))
        lays.append(lay)
        ys.append(device_tensor(skipconv_get_y(lay.handle), lay.shape_out, dt))
        h, w = lay.info.ho, lay.info.wo
    linked = 0
    if link:
        for li, L in enumerate(wl.layers):
            if li == 0:
                continue
            sc = None if L.shortcut <= 0 else lays[L.shortcut - 1]
            try:
                lays[li].link(lays[li - 1], sc)
                linked += 1
            except SkipConvError as e:
                # only layers on the one-launch CUDA-core step with TMA footprints take links
                assert e.status == SKIPCONV_ERR_UNSUPPORTED, e
    return lays, ys, dt, linked


def snapshot(lay):
    mask, lst, cnt = lay.gate()
    return (lay.z().view(torch.int32).cpu(), lay.y().view(torch.int16 if lay.dtype == torch.bfloat16 else torch.int32).cpu(),
            mask.cpu(), lst.cpu(), cnt, lay.prev_input().cpu())


def run_frame(wl, lays, ys, x, only=None):
    stack = [x]
    out = []
    for li, L in enumerate(wl.layers):
        if only is not None and li >= only:
            break
        lays[li].step(stack[-1], None if L.shortcut < 0 else stack[L.shortcut])
        stack.append(ys[li])
        out.append(li)
    return out


@pytest.mark.parametrize("name", ["c2", "c3"])
def test_linked_stack_is_bitwise_the_unlinked_stack(name):
    wl = synth.make_workload(name)
    A, ya, dt, _ = build_stack(wl, link=False, key_interval={3: 11})
    B, yb, _, linked = build_stack(wl, link=True, key_interval={3: 11})
    assert linked >= len(wl.layers) - 2, linked
    frames = [torch.from_numpy(np.ascontiguousarray(wl.frames[t])).cuda().to(dt) for t in range(wl.T)]
    try:
        for t in range(wl.T):
            if t == 9:
                # the first layer steps twice before the rest: its change flags then describe only its
                # last step, so its consumer must read the whole frame
                run_frame(wl, A, ya, frames[t - 1], only=1)
                run_frame(wl, B, yb, frames[t - 1], only=1)
            run_frame(wl, A, ya, frames[t])
            run_frame(wl, B, yb, frames[t])
            for li in range(len(wl.layers)):
                sa, sb = snapshot(A[li]), snapshot(B[li])
                for what, u, v in zip(("z", "y", "mask", "list", "count", "x_prev"), sa, sb):
                    if isinstance(u, int):
                        assert u == v, "%s t=%d layer %d: %s %d vs %d" % (name, t, li, what, u, v)
                    else:
                        assert torch.equal(u, v), "%s t=%d layer %d: %s differs" % (name, t, li, what)
    finally:
        for lay in A + B:
            lay.close()


def test_link_checks():
    wl = synth.make_workload("c3")
    lays, ys, dt, _ = build_stack(wl, link=False)
    try:
        # shapes: expand's y is [1][64][64][240], expand's own x_t is [1][64][64][40]
        with pytest.raises(SkipConvError) as ei:
            lays[0].link(lays[0])
        assert ei.value.status == SKIPCONV_ERR_INVALID
        with pytest.raises(SkipConvError) as ei:
            lays[3].link(lays[0])       # mb1.expand takes 40 channels, mb0.expand's y has 240
        assert ei.value.status == SKIPCONV_ERR_INVALID
        with pytest.raises(SkipConvError) as ei:
            lays[2].link(None, lays[0])   # a shortcut link needs the x_t link
        assert ei.value.status == SKIPCONV_ERR_INVALID
        lays[1].link(lays[0])
        lays[1].link(None)
        # a tensor-core layer (no y kept, weight-stationary) takes no links
        tc = SkipConvLayer(1, 64, 64, 64, 64, k=3, block=8, eps=0.05, dtype="bf16", conv_path=2,
                           weights=torch.zeros((64, 64, 3, 3)))
        with pytest.raises(SkipConvError) as ei:
            tc.link(lays[0])
        assert ei.value.status in (SKIPCONV_ERR_UNSUPPORTED, SKIPCONV_ERR_INVALID)
        tc.close()
        # destroying a producer drops the link
        lays[1].link(lays[0])
        lays[0].close()
        x = torch.zeros(lays[1].shape_in, dtype=dt, device="cuda")
        lays[1].step(x)
        torch.cuda.synchronize()
    finally:
        for lay in lays:
            lay.close()
