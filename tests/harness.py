"""Test helpers: run the CUDA layer and the oracle side by side on the same
seeded frames and compare them at every frame.

Comparison rules (floating point decides the gate, so both sides' decisions
are compared where they are unique):
  * block mask: bit-exact, except blocks whose oracle block score lies within
    1e-5 relative of eps (an fp32 score there may fall on either side); for the
    Gumbel gate (Eq. 8), whose threshold sits at 0, except blocks whose
    decision is not fixed within the fp32 error bound of f (tests/margin.py);
    the inputs keep a margin of twice that band, so no block is excluded
    (run_single_layer and run_stack_teacher_forced assert it);
  * active list: as a set (atomics make the order unspecified), equal to the
    GPU's own mask and to the oracle's mask outside the excluded blocks;
  * z: max-abs error <= 1e-4 for fp32 layers, <= 2e-2 * RMS(z_oracle) for bf16
    layers, at every frame; locations of a block excluded at some frame are
    left out from that frame on (its recurrence may legitimately differ);
  * x_{t-1} held by the layer equals x_t bit for bit after every step.
"""
from __future__ import annotations

import numpy as np

from margin import EPS_BAND, block_max, gumbel_bound, gumbel_undecided, norm_band  # noqa: F401

TOL_F32_ABS = 1e-4
TOL_BF16_REL_RMS = 2e-2


def to_device(a: np.ndarray, dtype: str):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a, np.float32))
    if dtype == "bf16":
        t = t.to(torch.bfloat16)          # values are already bf16-exact: no rounding happens here
    return t.cuda().contiguous()


class Compare:
    """Accumulates per-frame comparison results of one layer."""

    def __init__(self, spec, dtype: str, name: str = ""):
        self.spec, self.dtype, self.name = spec, dtype, name
        self.excluded = np.zeros((spec.n, spec.nby, spec.nbx), bool)
        self.max_err = 0.0
        self.max_rel = 0.0
        self.frames = 0
        self.n_excluded_events = 0

    def frame(self, t, score, mask_ref, gpu_mask, gpu_list, gpu_count, z_ref, z_gpu, forced, band=None):
        """band: the blocks excluded from the mask comparison at this frame; by
        default those whose oracle block score lies within EPS_BAND of eps."""
        s = self.spec
        if not forced:
            if band is None:
                band = norm_band(s, score, EPS_BAND)
            self.n_excluded_events += int(band.sum())
            self.excluded |= band
        else:
            band = np.zeros_like(self.excluded)
        ok = ~band
        diff = (gpu_mask != mask_ref) & ok
        assert not diff.any(), "%s t=%d: %d block gates differ (e.g. %s)" % (
            self.name, t, int(diff.sum()), np.argwhere(diff)[:5].tolist())
        ids = np.flatnonzero(gpu_mask.reshape(-1))
        assert gpu_count == len(ids), "%s t=%d: count %d vs mask %d" % (self.name, t, gpu_count, len(ids))
        np.testing.assert_array_equal(np.sort(gpu_list), ids, err_msg="%s t=%d: list != mask" % (self.name, t))
        # z, excluding the footprint of excluded blocks
        keep = np.repeat(np.repeat(~self.excluded, s.block, axis=1), s.block, axis=2)[:, :s.ho, :s.wo]
        err = np.abs(z_gpu - z_ref)[keep]
        e = float(err.max()) if err.size else 0.0
        rms = float(np.sqrt(np.mean(z_ref ** 2))) if z_ref.size else 0.0
        self.max_err = max(self.max_err, e)
        self.max_rel = max(self.max_rel, e / rms if rms > 0 else 0.0)
        if self.dtype == "f32":
            assert e <= TOL_F32_ABS, "%s t=%d: max |dz| = %.3g > %.1g" % (self.name, t, e, TOL_F32_ABS)
        else:
            assert e <= TOL_BF16_REL_RMS * rms, "%s t=%d: max |dz| = %.3g > 2e-2 * rms %.3g" % (
                self.name, t, e, rms)
        self.frames += 1


def gpu_layer(spec, w, bias, dtype, act=0, emit_y=False, dense_mode=False, conv_path=0, gate=None, key_interval=0,
              phi=None, phi_bias=0.0):
    import torch
    from paper_2104_11487_gb300 import SkipConvLayer
    wt = torch.from_numpy(np.ascontiguousarray(w, np.float32))
    bt = None if bias is None else torch.from_numpy(np.ascontiguousarray(bias, np.float32))
    return SkipConvLayer(spec.n, spec.c_in, spec.c_out, spec.h, spec.w, k=spec.k, stride=spec.stride, pad=spec.pad,
                         groups=spec.groups, block=spec.block, eps=spec.eps,
                         gate=spec.gate if gate is None else gate, dtype=dtype, activation=act, emit_y=emit_y,
                         dense_mode=dense_mode, conv_path=conv_path, weights=wt, bias=bt, key_interval=key_interval,
                         gate_weights=None if phi is None else torch.from_numpy(np.ascontiguousarray(phi, np.float32)),
                         gate_bias=phi_bias)


def run_single_layer(spec, w, bias, frames, dtype, dense_mode=False, conv_path=0, check_prev=True, name="",
                     reset_at=(), emit_y=False, expect_fused=None, key_interval=0, ref_reset_at=(), phi=None,
                     phi_bias=0.0, max_excluded=0):
    """Drive one layer over `frames` (iterable of float32 [n,h,w,c] arrays) on
    both sides; returns the Compare record and the conv path used.
    expect_fused: None, or the info.fused value the layer must report (0 separate
    launches, 1 one cooperative tensor-core launch, 2 one launch with a CTA per
    tile of gate blocks).
    reset_at: frames before which both sides are reset; ref_reset_at: frames
    before which only the oracle is reset (the GPU layer resets itself through
    key_interval)."""
    import oracle
    ref = oracle.OracleLayer(spec, w, bias, dense_mode=dense_mode, phi=phi, phi_bias=phi_bias)
    gl = gpu_layer(spec, w, bias, dtype, dense_mode=dense_mode, conv_path=conv_path, emit_y=emit_y,
                   key_interval=key_interval, phi=phi, phi_bias=phi_bias)
    cmp = Compare(spec, dtype, name)
    try:
        if expect_fused is not None:
            assert gl.info.fused == int(expect_fused), "%s: fused=%d" % (name, gl.info.fused)
        for t, f in enumerate(frames):
            if t in reset_at:
                ref.reset()
                gl.reset()
            if t in ref_reset_at:
                ref.reset()
            forced = ref.key or dense_mode
            band = None
            if spec.gate == oracle.GATE_GUMBEL and not forced:
                r = np.asarray(f, np.float64) - ref.x_prev
                band = gumbel_undecided(spec, oracle.gumbel_scores(spec, r, phi, phi_bias),
                                        gumbel_bound(spec, r, phi, phi_bias), spec.eps)
            score, mask_ref = ref.step(f)
            xt = to_device(f, dtype)
            gl.step(xt)
            mask, lst, cnt = gl.gate()
            cmp.frame(t, score, mask_ref, mask.cpu().numpy(), lst.cpu().numpy(), cnt, ref.z,
                      gl.z().cpu().numpy().astype(np.float64), forced, band)
            if emit_y:
                y_gpu = gl.y().float().cpu().numpy().astype(np.float64)
                y_ref = oracle.layer_output(ref.z, None, 0, 2 if dtype == "bf16" else 1)
                rms = float(np.sqrt(np.mean(y_ref ** 2)))
                allowed = (TOL_BF16_REL_RMS * rms if dtype == "bf16" else TOL_F32_ABS) + np.abs(y_ref) * 2.0 ** -7
                assert (np.abs(y_gpu - y_ref) <= allowed).all(), "%s t=%d: y beyond tolerance" % (name, t)
            if check_prev:
                import torch
                assert torch.equal(gl.prev_input().view(torch.int16 if dtype == "bf16" else torch.int32),
                                   xt.view(torch.int16 if dtype == "bf16" else torch.int32)), \
                    "%s t=%d: x_{t-1} is not x_t after the step" % (name, t)
        assert gl.info.conv_path in (1, 2)
        assert cmp.n_excluded_events <= max_excluded, "%s: %d block decisions in the eps band" % (
            name, cmp.n_excluded_events)
        return cmp, gl.info.conv_path
    finally:
        gl.close()


def run_stack_teacher_forced(wl, T=None, conv_path=0, max_excluded=0):
    """Run every layer of a stack workload teacher-forced: each CUDA layer
    gets the oracle's input sequence (and shortcut) for that layer.  At most
    max_excluded block decisions (all layers) may fall in the band."""
    import oracle
    from oracle import LayerSpec
    frames = wl.frames if T is None else wl.frames[:T]
    T = len(frames)
    specs, refs, gls, cmps = [], [], [], []
    h, w = wl.h, wl.w
    for li, L in enumerate(wl.layers):
        spec = LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=h, w=w, k=L.k, stride=L.stride, pad=L.pad,
                         groups=L.groups, block=L.block, eps=L.eps)
        specs.append(spec)
        refs.append(oracle.OracleLayer(spec, wl.weights[li], wl.biases[li]))
        gls.append(gpu_layer(spec, wl.weights[li], wl.biases[li], wl.dtype, act=L.act, emit_y=True,
                             conv_path=conv_path))
        cmps.append(Compare(spec, wl.dtype, "%s/%s" % (wl.name, L.name)))
        h, w = spec.ho, spec.wo
    round_mode = 2 if wl.dtype == "bf16" else 1
    try:
        for t in range(T):
            stack = [np.asarray(frames[t], np.float64)]
            for li, L in enumerate(wl.layers):
                x = stack[-1]
                forced = refs[li].key
                score, mask_ref = refs[li].step(x)
                sc = None if L.shortcut < 0 else stack[L.shortcut]
                y_ref = oracle.layer_output(refs[li].z, sc, L.act, round_mode)
                gls[li].step(to_device(x, wl.dtype), None if sc is None else to_device(sc, wl.dtype))
                mask, lst, cnt = gls[li].gate()
                cmps[li].frame(t, score, mask_ref, mask.cpu().numpy(), lst.cpu().numpy(), cnt, refs[li].z,
                               gls[li].z().cpu().numpy().astype(np.float64), forced)
                # y = round_bf16(act(z [+ shortcut])): the z tolerance, plus one bf16 ulp of the value,
                # since z values a few fp32 ulps apart may round to neighbouring bf16 values
                y_gpu = gls[li].y().float().cpu().numpy().astype(np.float64)
                rms = float(np.sqrt(np.mean(y_ref ** 2)))
                allowed = TOL_BF16_REL_RMS * rms + np.abs(y_ref) * 2.0 ** -7 + 1e-30
                bad = np.abs(y_gpu - y_ref) > allowed
                assert not bad.any(), "%s t=%d: %d y values beyond tolerance (max err %.3g, rms %.3g)" % (
                    cmps[li].name, t, int(bad.sum()), float(np.abs(y_gpu - y_ref).max()), rms)
                stack.append(y_ref)
        excl = sum(c.n_excluded_events for c in cmps)
        assert excl <= max_excluded, "%s: %d block decisions in the eps band" % (wl.name, excl)
        return cmps, [g.info.conv_path for g in gls]
    finally:
        for g in gls:
            g.close()
