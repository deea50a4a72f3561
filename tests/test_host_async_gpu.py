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


@pytest.mark.parametrize("path,block,hw", [(0, 8, (32, 40)), (1, 8, (30, 37)), (1, 3, (19, 23))])
def test_sparse_host_result_rebuilds_z(path, block, hw):
    """skipconv_step_host_sparse_async: the open blocks of each step (count,
    ids, z~ values written straight into pinned host memory), applied to a
    host copy of z~ in order, keep that copy equal to the device's z~ after
    every step -- the whole frame at the key frame, then only what changed
    (Eq. 3).  Ragged frames give partial edge blocks; two result buffers
    alternate between steps while the pipeline runs ahead."""
    from paper_2104_11487_gb300 import skipconv_step_host_sparse_async
    n, c, T = 2, 64, 6
    h, w = hw
    v = np.stack([synth.moving_squares_video(71 + s, T, h, w, c, n_squares=2, size=6, speed=2, noise_std=0.01)
                  for s in range(n)], axis=1)
    frames = [torch.from_numpy(synth.round_to_bf16(v[t])).to(torch.bfloat16).pin_memory() for t in range(T)]
    rng = np.random.default_rng(3)
    wt = torch.from_numpy(synth.he_weights(rng, c, c, 3, bf16=True))
    lay = SkipConvLayer(n, c, c, h, w, k=3, block=block, eps=0.05, dtype="bf16", conv_path=path, weights=wt)
    try:
        nby, nbx = lay.info.nby, lay.info.nbx
        nblk = n * nby * nbx
        zb = [torch.full((nblk, block, block, c), -1.0, dtype=torch.float32).pin_memory() for _ in range(2)]
        lb = [torch.full((nblk,), -1, dtype=torch.int32).pin_memory() for _ in range(2)]
        cb = [torch.full((1,), -1, dtype=torch.int32).pin_memory() for _ in range(2)]
        z_host = np.zeros((n, nby * block, nbx * block, c), np.float32)
        counts = []
        for t in range(T):
            skipconv_step_host_sparse_async(lay.handle, frames[t], zb[t % 2], lb[t % 2], cb[t % 2])
            skipconv_sync(lay.handle)
            cnt = int(cb[t % 2][0])
            ids = lb[t % 2][:cnt].numpy()
            mask, _, dev_cnt = lay.gate()
            mask = mask.cpu().numpy().reshape(-1)
            assert sorted(ids.tolist()) == np.flatnonzero(mask).tolist(), \
                "step %d: ids differ from the gate (host count %d, device count %d, fused %d)" % (
                    t, cnt, dev_cnt, lay.info.fused)
            blocks = zb[t % 2][:cnt].numpy()
            for i, bid in enumerate(ids):
                bx, by, s = bid % nbx, (bid // nbx) % nby, bid // (nbx * nby)
                z_host[s, by * block:(by + 1) * block, bx * block:(bx + 1) * block] = blocks[i]
            z_dev = lay.z().cpu().numpy()
            assert np.array_equal(z_host[:, :lay.info.ho, :lay.info.wo], z_dev), "step %d: rebuilt z differs" % t
            # past the frame's edge the blocks carry zeros
            assert not z_host[:, lay.info.ho:].any() and not z_host[:, :, lay.info.wo:].any()
            counts.append(cnt)
        assert counts[0] == nblk and 0 < min(counts[1:]) < nblk
    finally:
        lay.close()


def test_sparse_host_result_needs_mapped_host_memory():
    from paper_2104_11487_gb300 import skipconv_step_host_sparse_async
    from paper_2104_11487_gb300._lib import SKIPCONV_ERR_INVALID, SkipConvError
    lay = SkipConvLayer(1, 16, 16, 16, 16, k=3, block=8, eps=0.05, dtype="bf16", weights=torch.zeros(16, 16, 3, 3))
    try:
        x = torch.zeros((1, 16, 16, 16), dtype=torch.bfloat16).pin_memory()
        zb_pageable = torch.empty((4, 8, 8, 16), dtype=torch.float32)
        lb = torch.empty(4, dtype=torch.int32).pin_memory()
        cb = torch.empty(1, dtype=torch.int32).pin_memory()
        with pytest.raises(SkipConvError) as ei:
            skipconv_step_host_sparse_async(lay.handle, x, zb_pageable, lb, cb)
        assert ei.value.status == SKIPCONV_ERR_INVALID
    finally:
        lay.close()
