"""The eps margin of parity inputs.

A block whose gate score lies within rounding distance of eps may be decided
either way by an fp32 kernel, so the parity tests exclude such blocks (the
band, tests/harness.py) and want inputs that have none.  The generators draw
inputs only; this module measures, with the oracle's fp64 scores, how many
gate decisions of an input sequence fall inside the generator margin, which is
twice the exclusion band:

  * norm gates (Eq. 5, Eq. 7): block score within MARGIN_REL = 2e-5 relative
    of eps (the exclusion band is 1e-5);
  * the Gumbel gate (Eq. 8): a block whose decision is not fixed once every
    location's f is widened by twice its fp32 error bound (gumbel_bound).

A sequence with no such decision has no excluded block at the tests' band.
"""
from __future__ import annotations

import numpy as np

import oracle
from oracle import GATE_GUMBEL, LayerSpec

EPS_BAND = 1e-5          # exclusion band of the parity comparison (relative to eps)
MARGIN_REL = 2e-5        # generator margin (relative to eps)
U32 = 2.0 ** -24         # unit roundoff of float32


def block_max(score: np.ndarray, b: int) -> np.ndarray:
    """Ceil-mode b x b block maximum of [n, ho, wo] (edge blocks partial)."""
    n, ho, wo = score.shape
    nby, nbx = -(-ho // b), -(-wo // b)
    pad = np.full((n, nby * b, nbx * b), -np.inf)
    pad[:, :ho, :wo] = score
    return pad.reshape(n, nby, b, nbx, b).max(axis=(2, 4))


def gamma(m: int) -> float:
    """gamma_m = m u / (1 - m u): the relative bound on the rounding error of
    m float32 operations in a row (a sum of m + 1 terms in any order, each
    term carrying its own rounding)."""
    return m * U32 / (1.0 - m * U32)


def gumbel_bound(spec: LayerSpec, r: np.ndarray, phi: np.ndarray, phi_bias: float) -> np.ndarray:
    """Per output location, a bound on |f_fp32 - f| for the Gumbel gate score
    f = b + sum_{c,kh,kw} phi r (Eq. 8) when a kernel forms r = x_t - x_{t-1}
    in float32 (one rounding), each product in float32 (one rounding) and
    sums the k_h*k_w*c_in products and the bias in float32 in any order:
        |f_fp32 - f| <= gamma_{N+2} * (|b| + sum |phi| |r|),  N = k_h k_w c_in,
    since every term picks up at most N + 2 relative roundings (standard
    forward error analysis of a recursive or tree summation)."""
    n_terms = spec.k * spec.k * spec.c_in
    mag = oracle.gumbel_scores(spec, np.abs(r), np.abs(phi), abs(float(phi_bias)))
    return gamma(n_terms + 2) * mag


def gumbel_undecided(spec: LayerSpec, f: np.ndarray, bound: np.ndarray, eps: float) -> np.ndarray:
    """Blocks whose decision max f > eps is not fixed when every location's
    f may lie anywhere in [f - bound, f + bound]."""
    b = spec.block
    surely_open = block_max(f - bound, b) > eps
    maybe_open = block_max(f + bound, b) > eps
    return maybe_open & ~surely_open


def norm_band(spec: LayerSpec, score: np.ndarray, rel: float) -> np.ndarray:
    """Blocks whose maximum norm score lies within `rel` (relative) of eps."""
    bm = block_max(score, spec.block)
    return np.abs(bm - spec.eps) <= rel * max(spec.eps, 1e-30)


def layer_band_events(spec: LayerSpec, frames, w=None, phi=None, phi_bias: float = 0.0, key_frames=(0,),
                      key_interval: int = 0, flows=None) -> int:
    """Gate decisions of a single layer's input sequence (frames[t] float
    [n, h, w, c]) inside the generator margin.  Frame t is a key frame when t
    is in key_frames or, with key_interval K, when t is a multiple of K; a
    key frame decides no gate, and every later residual is x_t - x_{t-1}
    (warped by flows[t] when flows is given, Eq. 10)."""
    events = 0
    prev = None
    for t, f in enumerate(frames):
        f = np.asarray(f, np.float64)
        key = prev is None or t in key_frames or (key_interval > 0 and t % key_interval == 0)
        if not key:
            xp = prev if flows is None else oracle.warp(prev, flows[t])
            r = f - xp
            if spec.gate == GATE_GUMBEL:
                score = oracle.gumbel_scores(spec, r, phi, phi_bias)
                bound = gumbel_bound(spec, r, phi, phi_bias)
                events += int(gumbel_undecided(spec, score, 2.0 * bound, spec.eps).sum())
            else:
                score = oracle.gate_scores(spec, r, w)
                events += int(norm_band(spec, score, MARGIN_REL).sum())
        prev = f
    return events


def stack_band_events(wl) -> list:
    """Per layer of a stack workload, the gate decisions inside the generator
    margin when the oracle runs the stack over the workload's frames (each
    layer on the previous layers' bf16 outputs, as the teacher-forced parity
    test feeds them)."""
    specs, refs = [], []
    h, w = wl.h, wl.w
    for li, L in enumerate(wl.layers):
        spec = LayerSpec(n=wl.n, c_in=L.c_in, c_out=L.c_out, h=h, w=w, k=L.k, stride=L.stride, pad=L.pad,
                         groups=L.groups, block=L.block, eps=L.eps)
        specs.append(spec)
        refs.append(oracle.OracleLayer(spec, wl.weights[li], wl.biases[li]))
        h, w = spec.ho, spec.wo
    round_mode = 2 if wl.dtype == "bf16" else 1
    events = [0] * len(wl.layers)
    for t in range(len(wl.frames)):
        stack = [np.asarray(wl.frames[t], np.float64)]
        for li, L in enumerate(wl.layers):
            forced = refs[li].key
            score, _ = refs[li].step(stack[-1])
            if not forced:
                events[li] += int(norm_band(specs[li], score, MARGIN_REL).sum())
            sc = None if L.shortcut < 0 else stack[L.shortcut]
            stack.append(oracle.layer_output(refs[li].z, sc, L.act, round_mode))
    return events
