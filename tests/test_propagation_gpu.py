"""Stack propagation (skipconv_link_inputs): a linked layer skips the tiles
whose inputs did not change, and must produce exactly what the unlinked
layer produces -- z, y, gate masks, open-block lists and the committed
x_{t-1}, bit for bit, at every layer and frame of the c2 (pose-like) and c3
(MBConv-like) stacks run free (each layer on the previous layer's y on the
device), including key frames in the middle and a producer that steps twice
between two steps of its consumer.

The linked stack is also held to the oracle: at every layer and frame an
oracle layer steps on exactly the inputs the linked GPU layer received (its
producer's y, and the shortcut, copied to the host), and its gate masks,
lists, z~ and y are compared at the harness tolerances.  Unchanged locations
of a linked layer's input are the paper's copied outputs of the layer before
(Sec. 3.1), so this checks that a tile skipped for an unchanged input is what
the recurrence computes there."""
import numpy as np
import pytest
import torch

import oracle
import synth
from harness import TOL_BF16_REL_RMS, Compare
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


KEY_INTERVAL = {3: 11}      # layer 3 takes key frames at its steps 11 and 22 (Table 4)


class OracleStack:
    """One oracle layer per GPU layer, stepped on the inputs the GPU layers
    received (host copies of their device inputs)."""

    def __init__(self, wl):
        self.wl, self.refs, self.cmps, self.specs = wl, [], [], []
        h, w = wl.h, wl.w
        for li, L in enumerate(wl.layers):
            spec = oracle.LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=h, w=w, k=L.k, stride=L.stride,
                                    pad=L.pad, groups=L.groups, block=L.block, eps=L.eps)
            self.specs.append(spec)
            self.refs.append(oracle.OracleLayer(spec, wl.weights[li], wl.biases[li]))
            self.cmps.append(Compare(spec, wl.dtype, "%s/%s linked" % (wl.name, L.name)))
            h, w = spec.ho, spec.wo
        self.steps = [0] * len(wl.layers)

    def step(self, t, li, lay, x_host, sc_host):
        L = self.wl.layers[li]
        ki = KEY_INTERVAL.get(li, 0)
        if ki and self.steps[li] > 0 and self.steps[li] % ki == 0:
            self.refs[li].reset()
        self.steps[li] += 1
        ref = self.refs[li]
        forced = ref.key
        score, mask_ref = ref.step(x_host)
        mask, lst, cnt = lay.gate()
        self.cmps[li].frame(t, score, mask_ref, mask.cpu().numpy(), lst.cpu().numpy(), cnt, ref.z,
                            lay.z().cpu().numpy().astype(np.float64), forced)
        y_ref = oracle.layer_output(ref.z, sc_host, L.act, 2 if self.wl.dtype == "bf16" else 1)
        y_gpu = lay.y().float().cpu().numpy().astype(np.float64)
        rms = float(np.sqrt(np.mean(y_ref ** 2)))
        allowed = TOL_BF16_REL_RMS * rms + np.abs(y_ref) * 2.0 ** -7 + 1e-30
        keep = np.repeat(np.repeat(~self.cmps[li].excluded, L.block, axis=1), L.block, axis=2)
        keep = keep[:, :y_ref.shape[1], :y_ref.shape[2], None]
        bad = (np.abs(y_gpu - y_ref) > allowed) & keep
        assert not bad.any(), "%s t=%d: %d y values beyond tolerance" % (self.cmps[li].name, t, int(bad.sum()))


def host(x):
    return None if x is None else x.float().cpu().numpy().astype(np.float64)


def run_frame_checked(wl, lays, ys, x, ost, t, only=None):
    """run_frame, with every layer's inputs copied to the host and the oracle
    stepped on them right after the GPU layer stepped."""
    stack = [x]
    for li, L in enumerate(wl.layers):
        if only is not None and li >= only:
            break
        x_in = host(stack[-1])
        sc_dev = None if L.shortcut < 0 else stack[L.shortcut]
        sc_in = host(sc_dev)
        lays[li].step(stack[-1], sc_dev)
        ost.step(t, li, lays[li], x_in, sc_in)
        stack.append(ys[li])


# c2 and c3 run one wave of CTAs per layer, where the library reads the whole frame even when
# linked; dw3 (three depthwise layers on 8 streams of 128x128) runs several waves, where the links
# are used and tiles are skipped
STACKS = {"c2": {}, "c3": {}, "dw3": {"T": 12, "c": 64}}


@pytest.mark.parametrize("name", sorted(STACKS))
def test_linked_stack_is_bitwise_the_unlinked_stack(name):
    wl = synth.make_workload(name, **STACKS[name])
    A, ya, dt, _ = build_stack(wl, link=False, key_interval=KEY_INTERVAL)
    B, yb, _, linked = build_stack(wl, link=True, key_interval=KEY_INTERVAL)
    assert linked >= len(wl.layers) - 2, linked
    ost = OracleStack(wl)
    src = (wl.frames[t] for t in range(wl.T)) if isinstance(wl.frames, np.ndarray) else (f for _, f in wl.frames)
    frames = [torch.from_numpy(np.ascontiguousarray(f)).cuda().to(dt) for f in src]
    try:
        for t in range(wl.T):
            if t == 9:
                # the first layer steps twice before the rest: its change flags then describe only its
                # last step, so its consumer must read the whole frame
                run_frame(wl, A, ya, frames[t - 1], only=1)
                run_frame_checked(wl, B, yb, frames[t - 1], ost, t, only=1)
            run_frame(wl, A, ya, frames[t])
            run_frame_checked(wl, B, yb, frames[t], ost, t)
            for li in range(len(wl.layers)):
                sa, sb = snapshot(A[li]), snapshot(B[li])
                for what, u, v in zip(("z", "y", "mask", "list", "count", "x_prev"), sa, sb):
                    if isinstance(u, int):
                        assert u == v, "%s t=%d layer %d: %s %d vs %d" % (name, t, li, what, u, v)
                    else:
                        assert torch.equal(u, v), "%s t=%d layer %d: %s differs" % (name, t, li, what)
        # the inputs here are the GPU layers' own outputs, so no seed can keep them off eps: a block decided
        # within the band is reported (and left out of the comparison from then on), at most two in all
        excl = sum(c.n_excluded_events for c in ost.cmps)
        assert excl <= 2, "%s: %d block decisions in the eps band" % (name, excl)
        assert all(c.frames == wl.T + (1 if li == 0 else 0) for li, c in enumerate(ost.cmps))
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
