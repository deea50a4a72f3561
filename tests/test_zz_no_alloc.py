"""skipconv_gate_noalloc (the allocation-free gate entry point) against the
oracle's block gate and against the gate that skipconv_step computes, through
the C ABI, on two steps in a row.

The file name sorts last so that this test also runs after every other GPU
test in one session; it passes alone as well.  Masks and open-block sets must
agree bit for bit with the oracle's, except blocks whose fp64 oracle score
lies within 1e-5 relative of the threshold (an fp32 sum there may fall on
either side; the inputs keep twice that margin, so there are none).
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from synth.video import block_perturbation_video, moving_squares_video

from harness import EPS_BAND, block_max

pytestmark = pytest.mark.gpu

GATE_MEAN, GATE_SUM = 0, 1

# name, n, h, w, c, k, stride, pad, block, eps, gate, dtype, video
CASES = [
    ("bf16_c64_b8_blocks", 2, 64, 64, 64, 3, 1, 1, 8, 0.05, GATE_MEAN, "bf16", "blocks"),
    ("f32_c32_b1_squares", 1, 48, 40, 32, 3, 1, 1, 1, 0.05, GATE_MEAN, "f32", "squares"),
    ("f32_c3_stride2_ragged_sum", 2, 37, 29, 3, 3, 2, 1, 4, 1.0, GATE_SUM, "f32", "squares"),
]


def _frames(case):
    name, n, h, w, c, k, stride, pad, block, eps, gate, dtype, video = case
    if video == "blocks":
        it = block_perturbation_video(17, 3, n, h, w, c, block, 5, bf16=(dtype == "bf16"))
        return np.stack([np.array(f, np.float32) for _, f in it])   # the generator reuses its frame buffer
    v = np.stack([moving_squares_video(31 + s, 3, h, w, c, n_squares=3, size=8, speed=3, noise_std=0.01)
                  for s in range(n)], axis=1)
    return v.astype(np.float32)


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_noalloc_gate_matches_the_oracle_and_the_step_gate(case):
    import torch
    from paper_2104_11487_gb300 import SkipConvLayer, skipconv_gate_noalloc
    name, n, h, w, c, k, stride, pad, block, eps, gate, dtype, video = case
    frames = _frames(case)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    dev = [torch.from_numpy(f).to(tdt).cuda().contiguous() for f in frames]
    rng = np.random.default_rng(5)
    wts = (rng.standard_normal((c, c, k, k)) * 0.1).astype(np.float32)
    layer = SkipConvLayer(n, c, c, h, w, k=k, stride=stride, pad=pad, block=block, eps=eps, gate=gate,
                          dtype=dtype, weights=torch.from_numpy(wts))
    nby, nbx = layer.info.nby, layer.info.nbx
    mask = torch.full((n, nby, nbx), 7, dtype=torch.uint8, device="cuda")
    lst = torch.full((n * nby * nbx,), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    spec = oracle.LayerSpec(n=n, c_in=c, c_out=c, h=h, w=w, k=k, stride=stride, pad=pad, block=block, eps=eps,
                            gate=gate)
    thr = eps * c * k * k if gate == GATE_MEAN else eps

    layer.step(dev[0])                       # key frame
    checked = 0
    for t in (1, 2):                         # two calls in a row
        layer.step(dev[t])
        m_ref, l_ref, c_ref = layer.gate()
        stream = torch.cuda.current_stream()
        skipconv_gate_noalloc(layer.params, dev[t], dev[t - 1], mask, lst, cnt, stream.cuda_stream)
        torch.cuda.synchronize()
        m_ref = m_ref.cpu().numpy()
        m_new = mask.cpu().numpy()
        count = int(cnt.item())
        ids = np.sort(lst[:count].cpu().numpy())

        score = oracle.gate_scores(spec, frames[t].astype(np.float64) - frames[t - 1].astype(np.float64))
        sum_score = score * (c * k * k) if gate == GATE_MEAN else score
        band = np.abs(block_max(sum_score, block) - thr) <= EPS_BAND * thr
        assert not band.any(), "%s t=%d: %d blocks in the eps band" % (name, t, int(band.sum()))
        ok = ~band
        m_oracle = oracle.block_gate(spec, score)
        assert np.array_equal(m_new[ok], m_oracle[ok]), "%s t=%d: masks differ from the oracle's" % (name, t)
        assert np.array_equal(ids, np.flatnonzero(m_oracle.ravel())), "%s t=%d: open set != oracle's" % (name, t)
        assert np.array_equal(m_new[ok], m_ref[ok]), "%s t=%d: masks differ" % (name, t)
        assert set(np.unique(m_new)) <= {0, 1}
        assert np.array_equal(ids, np.flatnonzero(m_new.ravel())), "%s t=%d: list != mask" % (name, t)
        assert len(set(ids.tolist())) == count
        if not band.any():
            assert count == c_ref and np.array_equal(ids, l_ref.cpu().numpy())
        checked += int(ok.sum())
    assert checked > 0
    layer.close()


def test_noalloc_rejects_oversize_and_output_gate():
    import torch
    from paper_2104_11487_gb300 import skipconv_gate_noalloc
    from paper_2104_11487_gb300._lib import SkipConvError
    from paper_2104_11487_gb300._lib import BF16, F32, Params, SKIPCONV_ERR_INVALID, SKIPCONV_ERR_UNSUPPORTED
    x = torch.zeros(16, dtype=torch.float32, device="cuda")
    m = torch.zeros(16, dtype=torch.uint8, device="cuda")
    lst = torch.zeros(16, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
    # n*h*w one above the static scratch capacity (1 << 20 pixels): rejected before any launch
    big = Params(1, 8, 8, 1025, 1024, 3, 3, 1, 1, 1, 8, 0.05, GATE_MEAN, BF16, 0, 0, 0, 0)
    with pytest.raises(SkipConvError) as ei:
        skipconv_gate_noalloc(big, x, x, m, lst, cnt, None)
    assert ei.value.status == SKIPCONV_ERR_INVALID and "scratch" in str(ei.value)
    outg = Params(1, 8, 8, 4, 4, 3, 3, 1, 1, 1, 2, 0.05, 2, F32, 0, 0, 0, 0)
    with pytest.raises(SkipConvError) as ei:
        skipconv_gate_noalloc(outg, x, x, m, lst, cnt, None)
    assert ei.value.status == SKIPCONV_ERR_UNSUPPORTED


def test_noalloc_calls_take_no_device_memory():
    """After the first call (the per-device set-up), further calls leave the
    device's free memory unchanged."""
    import torch
    from paper_2104_11487_gb300 import skipconv_gate_noalloc
    from paper_2104_11487_gb300._lib import BF16, Params
    n, h, w, c = 2, 64, 64, 64
    p = Params(n, c, c, h, w, 3, 3, 1, 1, 1, 8, 0.05, GATE_MEAN, BF16, 0, 0, 0, 0)
    g = torch.Generator(device="cuda").manual_seed(3)
    a = torch.rand((n, h, w, c), generator=g, device="cuda").to(torch.bfloat16)
    b = torch.rand((n, h, w, c), generator=g, device="cuda").to(torch.bfloat16)
    m = torch.zeros((n, 8, 8), dtype=torch.uint8, device="cuda")
    lst = torch.zeros(n * 64, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    skipconv_gate_noalloc(p, a, b, m, lst, cnt, s)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(5):
        skipconv_gate_noalloc(p, a, b, m, lst, cnt, s)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert int(cnt.item()) == n * 64          # uniform random frames: every block open
