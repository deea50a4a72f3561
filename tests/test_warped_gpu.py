"""Warped residuals (Sec. 3.4, Eq. 10-11) on the GPU against the oracle:
r_t = x_t - T(x_{t-1}) and z~_t = T~(z~_{t-1}) + g (.) (w * r_t), T and T~
bilinear with a per-pixel flow.  Masks and lists exact outside the eps band,
z within the stated tolerances, y (with and without a shortcut), and the
committed x_{t-1} bit-exactly, at every frame; the flows are smooth
fractional fields that change per frame.  The cases cover the staged form's
warped variant (dense, depthwise, 1x1, several tiles with ragged edges) and
the general form (channel counts off the 16-byte vectors)."""
import numpy as np
import pytest
import torch

import synth
from harness import TOL_BF16_REL_RMS, TOL_F32_ABS, Compare, gpu_layer, to_device
from oracle import LayerSpec, OracleLayer, layer_output

pytestmark = pytest.mark.gpu

CASES = [
    # name, n, h, w, c_in, c_out, k, groups, block, dtype, conv_path, shortcut
    ("f32_b1", 1, 20, 18, 8, 8, 3, 1, 1, "f32", 0, False),
    ("bf16_b8_staged_layer", 2, 32, 40, 32, 32, 3, 1, 8, "bf16", 1, False),
    ("bf16_b8_shortcut", 2, 40, 36, 32, 32, 3, 1, 8, "bf16", 1, True),
    ("bf16_depthwise_b4", 1, 24, 24, 16, 16, 3, 16, 4, "bf16", 0, False),
    ("bf16_1x1_b4", 1, 16, 20, 24, 16, 1, 1, 4, "bf16", 0, False),
    # channel counts off the 16-byte vectors: the general form, and the scalar warp of z
    ("bf16_general_c12", 1, 18, 22, 12, 16, 3, 1, 2, "bf16", 1, True),
    ("f32_general_c6", 1, 14, 14, 6, 6, 3, 1, 2, "f32", 1, False),
]


def flows(rng, T, n, h, w):
    """Smooth fractional flow fields: a per-frame global shift plus a gentle wave."""
    yy, xx = np.meshgrid(np.arange(h), np.arange(w), indexing="ij")
    out = []
    for t in range(T):
        f = np.zeros((n, h, w, 2), np.float32)
        for s in range(n):
            gy, gx = rng.uniform(-1.5, 1.5, 2)
            f[s, ..., 0] = gy + 0.4 * np.sin(xx / 5.0 + t)
            f[s, ..., 1] = gx + 0.4 * np.cos(yy / 7.0 - t)
        out.append(f)
    return out


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_warped_steps_match_the_oracle(case):
    name, n, h, w, c_in, c_out, k, groups, block, dtype, path, with_sc = case
    rng = np.random.default_rng(500 + block)
    pad = (k - 1) // 2
    spec = LayerSpec(n=n, c_in=c_in, c_out=c_out, h=h, w=w, k=k, stride=1, pad=pad, groups=groups, block=block,
                     eps=0.05)
    v = np.stack([synth.moving_squares_video(91 + s, 6, h, w, c_in, n_squares=2, size=6, speed=2, noise_std=0.01)
                  for s in range(n)], axis=1)
    frames = synth.round_to_bf16(v) if dtype == "bf16" else v.astype(np.float32)
    wts = synth.he_weights(rng, c_out, c_in // groups, k, bf16=dtype == "bf16")
    b = (rng.standard_normal(c_out) * 0.1).astype(np.float32)
    b = synth.round_to_bf16(b) if dtype == "bf16" else b
    ref = OracleLayer(spec, wts, b)
    gl = gpu_layer(spec, wts, b, dtype, emit_y=True, conv_path=path)
    cmp = Compare(spec, dtype, name)
    fl = flows(rng, len(frames), n, h, w)
    try:
        assert gl.info.fused == 2
        for t in range(len(frames)):
            forced = ref.key
            score, mask_ref = ref.step_warped(frames[t], fl[t].astype(np.float64))
            xt = to_device(frames[t], dtype)
            sc = None
            if with_sc:
                sc = rng.standard_normal((n, h, w, c_out)).astype(np.float32) * 0.5
                sc = synth.round_to_bf16(sc) if dtype == "bf16" else sc
            gl.step_warped(xt, torch.from_numpy(fl[t]).cuda(), None if sc is None else to_device(sc, dtype))
            mask, lst, cnt = gl.gate()
            cmp.frame(t, score, mask_ref, mask.cpu().numpy(), lst.cpu().numpy(), cnt, ref.z,
                      gl.z().cpu().numpy().astype(np.float64), forced)
            y_gpu = gl.y().float().cpu().numpy().astype(np.float64)
            y_ref = layer_output(ref.z, sc, 0, 2 if dtype == "bf16" else 1)
            rms = float(np.sqrt(np.mean(y_ref ** 2)))
            allowed = (TOL_BF16_REL_RMS * rms if dtype == "bf16" else TOL_F32_ABS) + np.abs(y_ref) * 2.0 ** -7
            assert (np.abs(y_gpu - y_ref) <= allowed).all(), "%s t=%d: y beyond tolerance" % (name, t)
            view = torch.int16 if dtype == "bf16" else torch.int32
            assert torch.equal(gl.prev_input().view(view), xt.view(view)), "%s t=%d: x_{t-1} is not x_t" % (name, t)
        # warping moves errors between locations: the data keeps every block away from eps
        assert cmp.n_excluded_events == 0
        assert cmp.frames == len(frames)
    finally:
        gl.close()


def test_warped_step_needs_a_same_size_cuda_core_layer():
    from paper_2104_11487_gb300._lib import SKIPCONV_ERR_UNSUPPORTED, SkipConvError
    spec = LayerSpec(n=1, c_in=8, c_out=8, h=16, w=16, k=3, stride=2, pad=1, block=2, eps=0.05)
    rng = np.random.default_rng(1)
    gl = gpu_layer(spec, synth.he_weights(rng, 8, 8, 3, bf16=False), None, "f32")
    try:
        with pytest.raises(SkipConvError) as ei:
            gl.step_warped(torch.zeros((1, 16, 16, 8), device="cuda"), torch.zeros((1, 16, 16, 2), device="cuda"))
        assert ei.value.status == SKIPCONV_ERR_UNSUPPORTED
    finally:
        gl.close()
