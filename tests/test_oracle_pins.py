"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test ties the oracle to something other than itself: hand-derived
worked examples (tests/golden), library routines that compute a special case
(torch conv2d / max_pool2d, scipy correlate), closed forms (Eq. 2 with every
gate open), invariants (zero residual, linearity, Young's inequality, Eq. 6)
and an independent brute-force formulation on tiny inputs.
"""
import json
import os

import numpy as np
import pytest
import scipy.signal
import torch
import torch.nn.functional as F

import oracle
from oracle import GATE_INPUT_MEAN, GATE_INPUT_SUM, GATE_OUTPUT, LayerSpec, OracleLayer

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
GATES = {"input_mean": GATE_INPUT_MEAN, "input_sum": GATE_INPUT_SUM, "output": GATE_OUTPUT}


def torch_conv(spec: LayerSpec, w, x, bias=None):
    """Library dense convolution (cross-correlation), NHWC in/out, float64."""
    xt = torch.from_numpy(np.ascontiguousarray(x, np.float64)).permute(0, 3, 1, 2)
    wt = torch.from_numpy(np.ascontiguousarray(w, np.float64))
    bt = None if bias is None else torch.from_numpy(np.asarray(bias, np.float64))
    z = F.conv2d(xt, wt, bt, stride=spec.stride, padding=spec.pad, groups=spec.groups)
    return z.permute(0, 2, 3, 1).numpy()


def rand_layer(rng, spec):
    w = rng.standard_normal((spec.c_out, spec.c_in // spec.groups, spec.k, spec.k))
    b = rng.standard_normal(spec.c_out)
    return w, b


SHAPES = [
    LayerSpec(n=2, c_in=3, c_out=4, h=9, w=7, k=3, stride=1, pad=1, block=2),
    LayerSpec(n=1, c_in=4, c_out=5, h=11, w=10, k=3, stride=2, pad=1, block=3),
    LayerSpec(n=1, c_in=6, c_out=6, h=8, w=9, k=3, stride=1, pad=1, groups=6, block=4),
    LayerSpec(n=2, c_in=4, c_out=6, h=6, w=6, k=1, stride=1, pad=0, groups=2, block=4),
    LayerSpec(n=1, c_in=2, c_out=3, h=7, w=5, k=5, stride=1, pad=2, block=1),
]


# ------------------------------------------------------------ golden examples
def test_golden_center_pixel():
    g = json.load(open(os.path.join(GOLDEN, "input_norm_center_pixel.json")))
    L = g["layer"]
    frames = [np.array(f, np.float64)[None] for f in g["frames_hwc"]]
    for case in g["cases"]:
        spec = LayerSpec(L["n"], L["c_in"], L["c_out"], L["h"], L["w"], L["k"], L["stride"],
                         L["pad"], L["groups"], L["block"], case["eps"], GATES[case["gate"]])
        lay = OracleLayer(spec, np.array(g["weights"], np.float64), np.array(g["bias"]))
        s1, m1 = lay.step(frames[0])
        assert m1.all(), "first frame after reset is a key frame"
        np.testing.assert_array_equal(lay.z[0, :, :, 0], 0.5)
        s2, m2 = lay.step(frames[1])
        np.testing.assert_allclose(s2[0], case["score_t2"], rtol=1e-15)
        np.testing.assert_array_equal(m2[0], np.array(case["mask_t2"]))
        np.testing.assert_array_equal(lay.z[0, :, :, 0], np.array(case["z_t2"]))


def test_golden_block_ceil_edges():
    g = json.load(open(os.path.join(GOLDEN, "block_gate_ceil_edges.json")))
    L = g["layer"]
    spec = LayerSpec(L["n"], L["c_in"], L["c_out"], L["h"], L["w"], L["k"], L["stride"], L["pad"],
                     L["groups"], L["block"], g["eps"])
    lay = OracleLayer(spec, np.array(g["weights"], np.float64), np.array(g["bias"]))
    for f, m, z in zip(g["frames_hw"], g["masks"], g["z_hw"]):
        _, mask = lay.step(np.array(f, np.float64)[None, :, :, None])
        np.testing.assert_array_equal(mask[0], np.array(m))
        np.testing.assert_array_equal(lay.z[0, :, :, 0], np.array(z))


def test_golden_stride2_support():
    g = json.load(open(os.path.join(GOLDEN, "stride2_support.json")))
    L = g["layer"]
    spec = LayerSpec(L["n"], L["c_in"], L["c_out"], L["h"], L["w"], L["k"], L["stride"], L["pad"],
                     L["groups"], L["block"], g["eps"])
    lay = OracleLayer(spec, np.array(g["weights"], np.float64), np.array(g["bias"]))
    lay.step(np.zeros((1, 5, 5, 1)))
    x = np.zeros((1, 5, 5, 1))
    x[0, g["pixel"][0], g["pixel"][1], 0] = 1.0
    score, _ = lay.step(x)
    np.testing.assert_allclose(score[0], np.array(g["score_t2"]), rtol=1e-15, atol=0)
    np.testing.assert_array_equal(lay.z[0, :, :, 0], np.array(g["z_t2"], np.float64))


# ---------------------------------------------------------------- closed forms
@pytest.mark.parametrize("si", range(len(SHAPES)))
def test_all_gates_open_equals_dense_conv(si):
    """Eq. 2: with every gate open (eps = 0 on generic data, or dense mode)
    the recurrence reproduces the standard convolution of every frame."""
    spec = SHAPES[si]
    rng = np.random.default_rng(si)
    w, b = rand_layer(rng, spec)
    for dense in (False, True):
        s = LayerSpec(**{**spec.__dict__, "eps": 0.0})
        lay = OracleLayer(s, w, b, dense_mode=dense)
        for t in range(5):
            x = rng.standard_normal((s.n, s.h, s.w, s.c_in))
            lay.step(x)
            np.testing.assert_allclose(lay.z, torch_conv(s, w, x, b), rtol=1e-10, atol=1e-10)
            np.testing.assert_allclose(lay.z, oracle.dense_conv(s, w, x, b), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("eps", [0.05, 10.0, 1e9])
def test_key_frame_is_dense_for_any_eps(eps):
    """Sec. 3.1: the first frame's residual is the frame itself and it is
    processed over the whole frame, so z_1 = w * x_1 + b for any threshold."""
    spec = LayerSpec(n=1, c_in=3, c_out=2, h=6, w=5, k=3, block=2, eps=eps)
    rng = np.random.default_rng(7)
    w, b = rand_layer(rng, spec)
    lay = OracleLayer(spec, w, b)
    x = rng.random((1, 6, 5, 3))
    _, mask = lay.step(x)
    assert mask.all()
    np.testing.assert_allclose(lay.z, torch_conv(spec, w, x, b), rtol=1e-12, atol=1e-12)
    np.testing.assert_array_equal(lay.x_prev, x)


def test_zero_residual_skips_and_keeps_state():
    """Sec. 3.1: a kernel support of zero residual has zero output, so the
    location is skipped and z~_{t-1} is kept exactly."""
    spec = LayerSpec(n=2, c_in=3, c_out=4, h=8, w=8, k=3, block=2, eps=0.0)
    rng = np.random.default_rng(3)
    w, b = rand_layer(rng, spec)
    lay = OracleLayer(spec, w, b)
    x = rng.random((2, 8, 8, 3))
    lay.step(x)
    z1 = lay.z.copy()
    score, mask = lay.step(x.copy())
    assert not mask.any()
    np.testing.assert_array_equal(score, 0.0)
    np.testing.assert_array_equal(lay.z, z1)


def test_linearity_of_update():
    """Eq. 2 rests on the linearity of w * r: with every gate open the update
    for a*r1 + r2 is a*(update for r1) + (update for r2)."""
    spec = LayerSpec(n=1, c_in=4, c_out=3, h=7, w=6, k=3, stride=2, block=2, eps=0.0)
    rng = np.random.default_rng(11)
    w, _ = rand_layer(rng, spec)
    r1, r2 = rng.standard_normal((2, 1, 7, 6, 4))
    a = -1.75

    def update(r):
        lay = OracleLayer(spec, w, None, dense_mode=True)
        lay.step(r)             # x_prev = 0, so the residual is r itself
        return lay.z

    np.testing.assert_allclose(update(a * r1 + r2), a * update(r1) + update(r2), rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------------- the gate
@pytest.mark.parametrize("si", range(len(SHAPES)))
def test_gate_score_is_local_l1_box_sum(si):
    """Eq. 5 with p = 1: the channel-summed |r| correlated with a k x k box
    (zero padding, the layer's stride) — computed here with scipy."""
    spec = SHAPES[si]
    rng = np.random.default_rng(100 + si)
    r = rng.standard_normal((spec.n, spec.h, spec.w, spec.c_in))
    for gate in (GATE_INPUT_MEAN, GATE_INPUT_SUM, GATE_OUTPUT):
        s = LayerSpec(**{**spec.__dict__, "gate": gate})
        w, _ = rand_layer(rng, s)
        got = oracle.gate_scores(s, r, w)
        for n in range(s.n):
            a = np.abs(r[n]).sum(axis=2)
            a = np.pad(a, s.pad)
            box = scipy.signal.correlate2d(a, np.ones((s.k, s.k)), mode="valid")[::s.stride, ::s.stride]
            box = box[:s.ho, :s.wo]
            if gate == GATE_INPUT_MEAN:
                box = box / (s.c_in * s.k * s.k)
            elif gate == GATE_OUTPUT:
                box = box * np.abs(w).sum()
            np.testing.assert_allclose(got[n], box, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("b,h,w", [(1, 5, 7), (2, 7, 9), (4, 9, 6), (8, 16, 13), (3, 3, 3)])
def test_block_gate_is_max_pool_ceil(b, h, w):
    """Sec. 3.2: max-pool with kernel and stride b of the pixel gate (ceil
    mode at ragged edges) — torch max_pool2d is the independent routine."""
    spec = LayerSpec(n=2, c_in=1, c_out=1, h=h, w=w, k=1, pad=0, block=b, eps=0.5)
    rng = np.random.default_rng(b * 100 + h)
    score = rng.random((2, h, w))
    mask = oracle.block_gate(spec, score)
    pix = torch.from_numpy((score > 0.5).astype(np.float64))[:, None]
    ref = F.max_pool2d(pix, b, b, ceil_mode=True)[:, 0].numpy().astype(np.uint8)
    np.testing.assert_array_equal(mask, ref)
    if b == 1:
        np.testing.assert_array_equal(mask, (score > 0.5).astype(np.uint8))
    assert oracle.block_gate(spec, score, force=True).all()


def test_output_norm_gate_bounds_skipped_update():
    """Eq. 6 with r = s = q = 1 gives |w * r| <= ||w||_1 ||r||_1 locally, so an
    Output-Norm gate (Eq. 7) that stays closed skips an update of at most eps
    at that location and channel."""
    spec = LayerSpec(n=1, c_in=3, c_out=4, h=10, w=9, k=3, block=1, eps=0.8, gate=GATE_OUTPUT)
    rng = np.random.default_rng(5)
    w, b = rand_layer(rng, spec)
    w *= 0.05
    lay = OracleLayer(spec, w, b)
    x = rng.random((1, 10, 9, 3))
    lay.step(x)
    closed_seen = 0
    for t in range(6):
        x_new = x + rng.standard_normal(x.shape) * 0.02 * (rng.random((1, 10, 9, 1)) < 0.3)
        r = x_new - x
        full_update = torch_conv(spec, w, r)
        z_before = lay.z.copy()
        score, mask = lay.step(x_new)
        closed = mask[0] == 0
        closed_seen += int(closed.sum())
        assert np.all(np.abs(full_update[0][closed]) <= spec.eps + 1e-12)
        np.testing.assert_array_equal(lay.z[0][closed], z_before[0][closed])
        np.testing.assert_allclose(lay.z[0][~closed], (z_before + full_update)[0][~closed], rtol=1e-12, atol=1e-12)
        x = x_new
    assert closed_seen > 0


def test_skip_error_bound_input_norm_mean():
    """A closed Input-Norm gate (mean mode) bounds the skipped update at a
    location by max|w| * c_in * k^2 * eps; the drift from the dense result
    stays within the sum of those bounds over the steps (Eq. 3 vs Eq. 2)."""
    spec = LayerSpec(n=1, c_in=4, c_out=3, h=12, w=12, k=3, block=2, eps=0.02)
    rng = np.random.default_rng(9)
    w, b = rand_layer(rng, spec)
    lay = OracleLayer(spec, w, b)
    x = rng.random((1, 12, 12, 4))
    lay.step(x)
    bound_per_step = np.abs(w).max() * spec.c_in * spec.k * spec.k * spec.eps
    for t in range(1, 8):
        x = x + rng.standard_normal(x.shape) * 0.01
        _, mask = lay.step(x)
        drift = np.abs(lay.z - torch_conv(spec, w, x, b)).max()
        assert drift <= t * bound_per_step + 1e-12
    assert drift > 0, "some residuals were skipped"


# ------------------------------------------------------------- brute force
def brute_force_sequence(spec: LayerSpec, w, b, frames):
    """Scatter formulation on tiny inputs: every input pixel of the residual
    pushes its contribution to each output that reads it; gates are found by
    enumerating each block's locations and their receptive fields."""
    ho, wo = spec.ho, spec.wo
    cpg, opg = spec.c_in // spec.groups, spec.c_out // spec.groups
    z = np.tile(np.asarray(b, np.float64), (spec.n, ho, wo, 1))
    prev = np.zeros_like(frames[0])
    masks = []
    for t, x in enumerate(frames):
        r = x - prev
        upd = np.zeros_like(z)
        recept = {}
        for n in range(spec.n):
            for y in range(spec.h):
                for xx in range(spec.w):
                    for kh in range(spec.k):
                        for kw in range(spec.k):
                            i, rem_i = divmod(y + spec.pad - kh, spec.stride)
                            j, rem_j = divmod(xx + spec.pad - kw, spec.stride)
                            if rem_i or rem_j or not (0 <= i < ho and 0 <= j < wo):
                                continue
                            recept.setdefault((n, i, j), []).append((y, xx))
                            for c in range(spec.c_in):
                                g = c // cpg
                                for o in range(g * opg, (g + 1) * opg):
                                    upd[n, i, j, o] += w[o, c - g * cpg, kh, kw] * r[n, y, xx, c]
        mask = np.zeros((spec.n, spec.nby, spec.nbx), np.uint8)
        for n in range(spec.n):
            for by in range(spec.nby):
                for bx in range(spec.nbx):
                    best = 0.0
                    for i in range(by * spec.block, min(ho, (by + 1) * spec.block)):
                        for j in range(bx * spec.block, min(wo, (bx + 1) * spec.block)):
                            tot = sum(abs(r[n, y, xx, c]) for (y, xx) in recept.get((n, i, j), [])
                                      for c in range(spec.c_in))
                            best = max(best, tot / (spec.c_in * spec.k * spec.k))
                    mask[n, by, bx] = 1 if (t == 0 or best > spec.eps) else 0
        for n in range(spec.n):
            for i in range(ho):
                for j in range(wo):
                    if mask[n, i // spec.block, j // spec.block]:
                        z[n, i, j] += upd[n, i, j]
        masks.append(mask)
        prev = x
    return z, masks


@pytest.mark.parametrize("stride,groups,block", [(1, 1, 1), (2, 1, 1), (1, 2, 2), (1, 1, 3)])
def test_brute_force_tiny(stride, groups, block):
    spec = LayerSpec(n=1, c_in=2, c_out=4 if groups == 2 else 3, h=5, w=5, k=3, stride=stride, pad=1,
                     groups=groups, block=block, eps=0.15)
    rng = np.random.default_rng(stride * 10 + groups + block)
    w, b = rand_layer(rng, spec)
    base = rng.random((1, 5, 5, 2))
    frames = [base]
    for t in range(2):
        f = frames[-1].copy()
        y0, x0 = rng.integers(0, 4, size=2)
        f[0, y0:y0 + 2, x0:x0 + 2, :] += rng.random((2, 2, 2))
        f += rng.standard_normal(f.shape) * 0.01
        frames.append(f)
    z_ref, masks_ref = brute_force_sequence(spec, w, b, frames)
    lay = OracleLayer(spec, w, b)
    for t, f in enumerate(frames):
        _, mask = lay.step(f)
        np.testing.assert_array_equal(mask, masks_ref[t])
    assert any(not m.all() for m in masks_ref[1:]), "the case must close some gates"
    np.testing.assert_allclose(lay.z, z_ref, rtol=1e-12, atol=1e-12)


# ---------------------------------------------------- storage and activations
def test_bf16_rounding_matches_library():
    rng = np.random.default_rng(0)
    v = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.3895e38, 1e-40])]).astype(np.float32)
    ref = torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy()
    got = oracle.round_bf16(v.astype(np.float64))
    np.testing.assert_array_equal(got, ref)


def test_layer_output_activations_match_library():
    rng = np.random.default_rng(1)
    z = rng.standard_normal(5000) * 3
    sc = rng.standard_normal(5000)
    zt, st = torch.from_numpy(z), torch.from_numpy(sc)
    np.testing.assert_allclose(oracle.layer_output(z, sc, oracle.ACT_RELU), F.relu(zt + st).numpy(), rtol=1e-15)
    np.testing.assert_allclose(oracle.layer_output(z, None, oracle.ACT_SILU), F.silu(zt).numpy(), rtol=1e-14)
    np.testing.assert_array_equal(oracle.layer_output(z, sc, oracle.ACT_NONE), z + sc)


def test_sampled_layer_matches_full_layer():
    spec = LayerSpec(n=2, c_in=4, c_out=5, h=10, w=9, k=3, block=3, eps=0.1)
    rng = np.random.default_rng(21)
    w, b = rand_layer(rng, spec)
    samples = np.array([[0, 0, 0], [1, 9, 8], [0, 4, 5], [1, 2, 7]], np.int32)
    full = OracleLayer(spec, w, b)
    samp = oracle.SampledOracleLayer(spec, w, samples, b)
    x = rng.random((2, 10, 9, 4))
    for t in range(5):
        _, m1 = full.step(x)
        m2 = samp.step(x)
        np.testing.assert_array_equal(m1, m2)
        np.testing.assert_array_equal(samp.z, full.z[samples[:, 0], samples[:, 1], samples[:, 2]])
        x = x.copy()
        x[:, t:t + 3, 1:4] += rng.random((2, 3, 3, 4))


# ------------------------------------------------------- Gumbel gate (Eq. 8)
@pytest.mark.parametrize("si", range(len(SHAPES)))
def test_gumbel_score_is_single_channel_conv(si):
    """f(r; phi) is a convolution with one output channel and the layer's
    kernel, stride and padding (plus its bias): torch's conv2d computes it."""
    s = SHAPES[si]
    spec = LayerSpec(n=s.n, c_in=s.c_in, c_out=s.c_out, h=s.h, w=s.w, k=s.k, stride=s.stride, pad=s.pad,
                     groups=s.groups, block=s.block, eps=0.0, gate=oracle.GATE_GUMBEL)
    rng = np.random.default_rng(300 + si)
    r = rng.standard_normal((spec.n, spec.h, spec.w, spec.c_in))
    phi = rng.standard_normal((spec.c_in, spec.k, spec.k))
    bias = 0.37
    ref = torch_conv(LayerSpec(n=spec.n, c_in=spec.c_in, c_out=1, h=spec.h, w=spec.w, k=spec.k, stride=spec.stride,
                               pad=spec.pad), phi[None], r, [bias])[..., 0]
    np.testing.assert_allclose(oracle.gumbel_scores(spec, r, phi, bias), ref, rtol=1e-12, atol=1e-12)


def test_gumbel_zero_residual_and_linearity():
    """r = 0 gives f = phi_bias everywhere (all gates open iff phi_bias > 0);
    f - phi_bias is linear in r."""
    spec = LayerSpec(n=1, c_in=3, c_out=2, h=7, w=6, k=3, block=2, eps=0.0, gate=oracle.GATE_GUMBEL)
    rng = np.random.default_rng(310)
    phi = rng.standard_normal((3, 3, 3))
    zero = np.zeros((1, 7, 6, 3))
    for b in (0.25, -0.25):
        f = oracle.gumbel_scores(spec, zero, phi, b)
        np.testing.assert_array_equal(f, np.full(f.shape, b))
        assert oracle.block_gate(spec, f).all() == (b > 0) and oracle.block_gate(spec, f).any() == (b > 0)
    r1, r2 = rng.standard_normal((2, 1, 7, 6, 3))
    a = 1.7
    lhs = oracle.gumbel_scores(spec, a * r1 + r2, phi, 0.0)
    rhs = a * oracle.gumbel_scores(spec, r1, phi, 0.0) + oracle.gumbel_scores(spec, r2, phi, 0.0)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("stride,block", [(1, 1), (2, 2), (1, 3)])
def test_gumbel_step_is_masked_dense_update(stride, block):
    """A Gumbel-gated step adds w * r exactly at the locations of blocks where
    max f > 0 (round(sigmoid(f)) = 1), brute force on a tiny layer."""
    spec = LayerSpec(n=1, c_in=2, c_out=3, h=6, w=5, k=3, stride=stride, pad=1, block=block, eps=0.0,
                     gate=oracle.GATE_GUMBEL)
    rng = np.random.default_rng(320 + stride + block)
    w, b = rand_layer(rng, spec)
    phi = rng.standard_normal((2, 3, 3))
    phi_b = -0.5
    frames = [rng.random((1, 6, 5, 2)) for _ in range(3)]
    lay = OracleLayer(spec, w, b, phi=phi, phi_bias=phi_b)
    z = torch_conv(spec, w, frames[0], b)
    lay.step(frames[0])                              # key frame
    np.testing.assert_allclose(lay.z, z, rtol=1e-12, atol=1e-12)
    closed = 0
    for t in (1, 2):
        r = frames[t] - frames[t - 1]
        f = torch_conv(LayerSpec(n=1, c_in=2, c_out=1, h=6, w=5, k=3, stride=stride, pad=1), phi[None], r,
                       [phi_b])[..., 0]
        ho, wo = f.shape[1:]
        nby, nbx = -(-ho // block), -(-wo // block)
        mask = np.zeros((1, nby, nbx), np.uint8)
        for by in range(nby):
            for bx in range(nbx):
                mask[0, by, bx] = f[0, by * block:by * block + block, bx * block:bx * block + block].max() > 0
        upd = torch_conv(spec, w, r)
        for i in range(ho):
            for j in range(wo):
                if mask[0, i // block, j // block]:
                    z[0, i, j] += upd[0, i, j]
        _, m = lay.step(frames[t])
        np.testing.assert_array_equal(m, mask)
        closed += int((mask == 0).sum())
        np.testing.assert_allclose(lay.z, z, rtol=1e-12, atol=1e-12)
    assert closed > 0, "the case must close some gates"


# ------------------------------------------------------- warped residuals (Eq. 10-11)
def test_warp_is_library_grid_sample():
    """T (bilinear, zero outside) equals torch's grid_sample with align_corners=True
    and zero padding, sampled at p + flow(p)."""
    rng = np.random.default_rng(71)
    n, h, w, c = 2, 7, 9, 3
    x = rng.standard_normal((n, h, w, c))
    flow = rng.uniform(-2.5, 2.5, (n, h, w, 2))
    got = oracle.warp(x, flow)
    yy, xx = np.meshgrid(np.arange(h), np.arange(w), indexing="ij")
    sy, sx = yy[None] + flow[..., 0], xx[None] + flow[..., 1]
    grid = np.stack([2 * sx / (w - 1) - 1, 2 * sy / (h - 1) - 1], axis=-1)      # (x, y) in [-1, 1]
    ref = F.grid_sample(torch.from_numpy(x).permute(0, 3, 1, 2), torch.from_numpy(grid), mode="bilinear",
                        padding_mode="zeros", align_corners=True).permute(0, 2, 3, 1).numpy()
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_warped_step_with_zero_flow_is_the_plain_step():
    """f(x) = x - x_{t-1} is the special case T = identity (Sec. 3.4): with a zero
    flow the warped step is the plain step, bit for bit."""
    rng = np.random.default_rng(72)
    spec = LayerSpec(n=2, c_in=3, c_out=4, h=9, w=8, k=3, block=2, eps=0.3)
    w, b = rand_layer(rng, spec)
    a, bb = OracleLayer(spec, w, b), OracleLayer(spec, w, b)
    zero = np.zeros((spec.n, spec.h, spec.w, 2))
    for t in range(5):
        x = rng.standard_normal((spec.n, spec.h, spec.w, spec.c_in)) * (0.2 if t else 1.0)
        s1, m1 = a.step(x)
        s2, m2 = bb.step_warped(x, zero)
        np.testing.assert_array_equal(m1, m2)
        np.testing.assert_array_equal(s1, s2)
        np.testing.assert_array_equal(a.z, bb.z)


@pytest.mark.parametrize("d", [(1, -2), (0, 3), (-1, 1)])
def test_warped_step_decodes_translations_exactly(d):
    """Eq. 11 with an equivariant warp: for an integer translation and every gate
    open, T~(z_{t-1}) + w * (x_t - T(x_{t-1})) = w * x_t + b at every location far
    enough from the border (the warp's zero fill and the convolution's padding
    differ near it), so the warped recurrence reproduces the dense output."""
    rng = np.random.default_rng(73)
    spec = LayerSpec(n=1, c_in=3, c_out=2, h=26, w=24, k=3, block=2, eps=0.0)
    w, b = rand_layer(rng, spec)
    lay = OracleLayer(spec, w, b)
    flow = np.zeros((1, spec.h, spec.w, 2))
    flow[..., 0], flow[..., 1] = d
    T = 4
    for t in range(T):
        x = rng.standard_normal((1, spec.h, spec.w, spec.c_in))
        _, m = lay.step_warped(x, flow)
        assert m.all()
    m = (T - 1) * max(abs(d[0]), abs(d[1])) + spec.pad + 1     # border band the error can reach after T steps
    ref = torch_conv(spec, w, x, b)
    inner = (slice(None), slice(m, spec.h - m), slice(m, spec.w - m))
    assert ref[inner].size > 0
    np.testing.assert_allclose(lay.z[inner], ref[inner], rtol=0, atol=1e-10 * np.abs(ref).max())
    # and the border does differ (the reading is not vacuous)
    assert np.abs(lay.z - ref).max() > 1e-6


def test_warped_step_brute_force_tiny():
    """The warped step written out with plain Python loops (bilinear weights of the
    four neighbours, zero outside; support sums; block max; masked update)."""
    rng = np.random.default_rng(74)
    spec = LayerSpec(n=1, c_in=2, c_out=2, h=6, w=5, k=3, block=2, eps=0.4)
    w, b = rand_layer(rng, spec)
    lay = OracleLayer(spec, w, b)
    x0 = rng.standard_normal((1, spec.h, spec.w, spec.c_in))
    lay.step(x0)
    z = lay.z.copy()
    xp = x0.copy()
    opened = []
    for t in range(3):
        # large changes in the top rows only, small flows: some blocks open, some stay closed
        amp = np.where(np.arange(spec.h)[None, :, None, None] < 2, 0.9, 0.02)
        x = xp + rng.standard_normal(xp.shape) * amp
        flow = rng.uniform(-0.25, 0.25, (1, spec.h, spec.w, 2))
        flow[0, :, :, 0] += 1.0 if t == 2 else 0.0      # and one frame shifted by a whole row

        def bil(a, y, xx, c):
            y0, x0_ = int(np.floor(y)), int(np.floor(xx))
            ay, ax = y - y0, xx - x0_
            v = 0.0
            for (yy, xq, wt) in ((y0, x0_, (1 - ay) * (1 - ax)), (y0, x0_ + 1, (1 - ay) * ax),
                                 (y0 + 1, x0_, ay * (1 - ax)), (y0 + 1, x0_ + 1, ay * ax)):
                if 0 <= yy < a.shape[1] and 0 <= xq < a.shape[2]:
                    v += wt * a[0, yy, xq, c]
            return v
        r = np.zeros_like(x)
        zw = np.zeros_like(z)
        for i in range(spec.h):
            for j in range(spec.w):
                fy, fx = flow[0, i, j]
                for c in range(spec.c_in):
                    r[0, i, j, c] = x[0, i, j, c] - bil(xp, i + fy, j + fx, c)
                for o in range(spec.c_out):
                    zw[0, i, j, o] = bil(z, i + fy, j + fx, o)
        score = np.zeros((spec.h, spec.w))
        delta = np.zeros_like(z)
        for i in range(spec.h):
            for j in range(spec.w):
                s = 0.0
                for kh in range(3):
                    for kw in range(3):
                        yy, xq = i + kh - 1, j + kw - 1
                        if 0 <= yy < spec.h and 0 <= xq < spec.w:
                            s += np.abs(r[0, yy, xq]).sum()
                            for o in range(spec.c_out):
                                delta[0, i, j, o] += (w[o, :, kh, kw] * r[0, yy, xq]).sum()
                score[i, j] = s / (spec.c_in * 9)
        mask = np.zeros((3, 3), bool)
        for by in range(3):
            for bx in range(3):
                mask[by, bx] = score[2 * by:2 * by + 2, 2 * bx:2 * bx + 2].max() > spec.eps
        z = zw + delta * np.repeat(np.repeat(mask, 2, 0), 2, 1)[None, :spec.h, :spec.w, None]
        xp = x
        s_o, m_o = lay.step_warped(x, flow)
        np.testing.assert_array_equal(m_o[0], mask)
        np.testing.assert_allclose(s_o[0], score, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(lay.z, z, rtol=1e-12, atol=1e-12)
        opened.append(int(mask.sum()))
    assert any(0 < k < 9 for k in opened), opened   # some frame mixes open and closed blocks
