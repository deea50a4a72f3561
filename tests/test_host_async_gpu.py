"""The pipelined host-buffer step (skipconv_step_host_async + skipconv_sync)
against the synchronous one (skipconv_step_host): the same frames from pinned
host memory give the same z at every step, each step's z landing in its own
host buffer although the copies of neighbouring steps overlap.  z is compared
within fp32 summation-order noise (the tensor-core epilogue adds its partial
sums into z by reduction, in no fixed order); the inputs committed as x_{t-1}
are compared bit for bit."""
import numpy as np
import pytest
import torch

import synth
from paper_2104_11487_gb300 import (SkipConvLayer, skipconv_step_host, skipconv_step_host_async,
                                    skipconv_sync)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("path", [0, 1])
def test_pipelined_host_steps_match_synchronous_ones(path):
    n, h, w, c, T = 2, 32, 40, 64, 7
    wl = synth.make_workload("c4", density=0.1, T=T, n=n, h=h, w=w, c=c)
    frames = [torch.from_numpy(np.ascontiguousarray(f, np.float32)).to(torch.bfloat16).pin_memory()
              for _, f in wl.frames]
    wt = torch.from_numpy(wl.weights[0])

    def layer():
        return SkipConvLayer(n, c, c, h, w, k=3, block=8, eps=0.05, dtype="bf16", conv_path=path, weights=wt)

    a, b = layer(), layer()
    try:
        za = [torch.empty((n, h, w, c), dtype=torch.float32).pin_memory() for _ in range(T)]
        zb = [torch.empty((n, h, w, c), dtype=torch.float32).pin_memory() for _ in range(T)]
        for t in range(T):
            skipconv_step_host(a.handle, frames[t], za[t])
        for t in range(T):
            skipconv_step_host_async(b.handle, frames[t], zb[t])
        skipconv_sync(b.handle)
        for t in range(T):
            scale = float(za[t].abs().max()) + 1e-30
            err = float((za[t] - zb[t]).abs().max())
            assert err <= 1e-5 * scale, "step %d: pipelined z differs by %.3g (max |z| %.3g)" % (t, err, scale)
        assert torch.equal(a.prev_input().view(torch.int16), b.prev_input().view(torch.int16))
        # no read-back, then a synchronous step after pipelined ones
        skipconv_step_host_async(b.handle, frames[0], None)
        skipconv_sync(b.handle)
        skipconv_step_host(b.handle, frames[1], zb[0])
    finally:
        a.close()
        b.close()
