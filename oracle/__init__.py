"""Skip-Convolution oracle (arXiv 2104.11487): a plain CPU reference of the
per-frame Skip-Conv layer step, in double precision.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference leg of ``bench.py`` may import this package.  It
shares no code with the CUDA library (``paper_2104_11487_gb300``) and never
imports it.

The arithmetic lives in ``skipconv_oracle.c`` (plain loops, one function per
step of the method, each citing its passage); this module builds it with gcc
and wraps it with ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "skipconv_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libskipconv_oracle.so")

GATE_INPUT_MEAN = 0
GATE_INPUT_SUM = 1
GATE_OUTPUT = 2
GATE_GUMBEL = 3
ACT_NONE = 0
ACT_RELU = 1
ACT_SILU = 2


def build(force: bool = False, openmp: bool = True) -> str:
    """Compile the oracle into a shared library (gcc, -O2, OpenMP if available)."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-lm"]
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    if openmp:
        r = subprocess.run(base[:1] + ["-fopenmp"] + base[1:] + ["-o", tmp],
                           capture_output=True, text=True)
        if r.returncode == 0:
            os.replace(tmp, _LIB_PATH)
            return _LIB_PATH
        sys.stderr.write("oracle: OpenMP build failed, building single-threaded\n" + r.stderr)
    subprocess.run(base + ["-o", tmp], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "n", "c_in", "c_out", "h", "w", "k_h", "k_w", "stride", "pad", "groups", "block", "gate")] + [
        ("eps", ctypes.c_double)]


_lib = None
_DP = ctypes.POINTER(ctypes.c_double)
_UP = ctypes.POINTER(ctypes.c_ubyte)
_IP = ctypes.POINTER(ctypes.c_int)


def lib():
    global _lib
    if _lib is None:
        path = build()
        L = ctypes.CDLL(path)
        PP = ctypes.POINTER(_Params)
        for name in ("oc_out_h", "oc_out_w", "oc_blocks_y", "oc_blocks_x"):
            getattr(L, name).argtypes = [PP]
            getattr(L, name).restype = ctypes.c_int
        L.oc_num_threads.restype = ctypes.c_int
        L.oc_set_num_threads.argtypes = [ctypes.c_int]
        L.oc_weight_l1.argtypes = [PP, _DP]
        L.oc_weight_l1.restype = ctypes.c_double
        L.oc_residual.argtypes = [PP, _DP, _DP, _DP]
        L.oc_gate_scores.argtypes = [PP, _DP, ctypes.c_double, _DP]
        L.oc_block_gate.argtypes = [PP, _DP, ctypes.c_int, _UP]
        L.oc_dense_conv.argtypes = [PP, _DP, _DP, _DP, _DP]
        L.oc_reset.argtypes = [PP, _DP, _DP, _DP]
        L.oc_gumbel_scores.argtypes = [PP, _DP, _DP, ctypes.c_double, _DP]
        L.oc_step.argtypes = [PP, _DP, _DP, ctypes.c_double, _DP, _DP, _DP, ctypes.c_int, _DP, _UP]
        L.oc_step.restype = ctypes.c_long
        L.oc_step_sampled.argtypes = [PP, _DP, _DP, ctypes.c_double, _DP, _DP, ctypes.c_int, _IP, _DP, ctypes.c_int,
                                      _UP]
        L.oc_step_sampled.restype = ctypes.c_long
        L.oc_warp.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _DP, _DP, _DP]
        L.oc_step_warped.argtypes = [PP, _DP, _DP, ctypes.c_double, _DP, _DP, _DP, _DP, ctypes.c_int, _DP, _UP]
        L.oc_step_warped.restype = ctypes.c_long
        L.oc_round_bf16.argtypes = [ctypes.c_double]
        L.oc_round_bf16.restype = ctypes.c_double
        L.oc_layer_output.argtypes = [ctypes.c_size_t, _DP, _DP, ctypes.c_int, ctypes.c_int, _DP]
        _lib = L
    return _lib


def _dp(a):
    return None if a is None else a.ctypes.data_as(_DP)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


@dataclass
class LayerSpec:
    """Shape of one Skip-Conv layer (names follow the paper's notation)."""
    n: int
    c_in: int
    c_out: int
    h: int
    w: int
    k: int = 3
    stride: int = 1
    pad: int = 1
    groups: int = 1
    block: int = 1
    eps: float = 0.05
    gate: int = GATE_INPUT_MEAN

    def params(self) -> _Params:
        return _Params(self.n, self.c_in, self.c_out, self.h, self.w, self.k, self.k,
                       self.stride, self.pad, self.groups, self.block, self.gate, float(self.eps))

    @property
    def ho(self) -> int:
        return (self.h + 2 * self.pad - self.k) // self.stride + 1

    @property
    def wo(self) -> int:
        return (self.w + 2 * self.pad - self.k) // self.stride + 1

    @property
    def nby(self) -> int:
        return -(-self.ho // self.block)

    @property
    def nbx(self) -> int:
        return -(-self.wo // self.block)


def num_threads() -> int:
    return lib().oc_num_threads()


def set_num_threads(t: int) -> None:
    lib().oc_set_num_threads(int(t))


def weight_l1(spec: LayerSpec, w) -> float:
    w = _f64(w)
    return lib().oc_weight_l1(ctypes.byref(spec.params()), _dp(w))


def gate_scores(spec: LayerSpec, r, w=None) -> np.ndarray:
    """Per-output-location gate score (Eq. 5 / Eq. 7) of a residual r [n,h,w,c_in]."""
    r = _f64(r)
    wl1 = weight_l1(spec, w) if spec.gate == GATE_OUTPUT else 0.0
    out = np.empty((spec.n, spec.ho, spec.wo), np.float64)
    lib().oc_gate_scores(ctypes.byref(spec.params()), _dp(r), wl1, _dp(out))
    return out


def gumbel_scores(spec: LayerSpec, r, phi, phi_bias: float = 0.0) -> np.ndarray:
    """Per-output-location Gumbel-gate score f(r; phi) (Eq. 8): a single-output-
    channel convolution of r [n,h,w,c_in] with phi [c_in, k, k] plus phi_bias."""
    r, phi = _f64(r), _f64(phi)
    assert phi.shape == (spec.c_in, spec.k, spec.k)
    out = np.empty((spec.n, spec.ho, spec.wo), np.float64)
    lib().oc_gumbel_scores(ctypes.byref(spec.params()), _dp(r), _dp(phi), float(phi_bias), _dp(out))
    return out


def block_gate(spec: LayerSpec, score, force: bool = False) -> np.ndarray:
    score = _f64(score)
    out = np.empty((spec.n, spec.nby, spec.nbx), np.uint8)
    lib().oc_block_gate(ctypes.byref(spec.params()), _dp(score), int(force),
                        out.ctypes.data_as(_UP))
    return out


def dense_conv(spec: LayerSpec, w, x, bias=None) -> np.ndarray:
    """Eq. 1: z = w * x (+ bias) at every output location, NHWC."""
    w, x = _f64(w), _f64(x)
    b = None if bias is None else _f64(bias)
    out = np.empty((spec.n, spec.ho, spec.wo, spec.c_out), np.float64)
    lib().oc_dense_conv(ctypes.byref(spec.params()), _dp(w), _dp(b), _dp(x), _dp(out))
    return out


def round_bf16(a) -> np.ndarray:
    """Nearest bfloat16 value of every element (ties to even), as float64."""
    return layer_output(a, None, ACT_NONE, 2)


def layer_output(z, shortcut=None, act: int = ACT_NONE, round_mode: int = 0) -> np.ndarray:
    """y = act(z [+ shortcut]) rounded to the storage precision (0 none, 1 fp32, 2 bf16)."""
    z = _f64(z)
    sc = None if shortcut is None else _f64(shortcut)
    y = np.empty_like(z)
    lib().oc_layer_output(z.size, _dp(z), _dp(sc), int(act), int(round_mode), _dp(y))
    return y


class OracleLayer:
    """Stateful Skip-Conv layer: holds x_{t-1} and z~_{t-1} (Eq. 3) in double."""

    def __init__(self, spec: LayerSpec, w, bias=None, dense_mode: bool = False, phi=None, phi_bias: float = 0.0):
        self.spec = spec
        self.w = _f64(w)
        assert self.w.shape == (spec.c_out, spec.c_in // spec.groups, spec.k, spec.k)
        self.phi = None if phi is None else _f64(phi)          # Gumbel gate function (gate mode 3)
        self.phi_bias = float(phi_bias)
        assert spec.gate != GATE_GUMBEL or (self.phi is not None and self.phi.shape == (spec.c_in, spec.k, spec.k))
        self.bias = None if bias is None else _f64(bias)
        self.dense_mode = bool(dense_mode)
        self.x_prev = np.zeros((spec.n, spec.h, spec.w, spec.c_in), np.float64)
        self.z = np.zeros((spec.n, spec.ho, spec.wo, spec.c_out), np.float64)
        self.reset()

    def reset(self) -> None:
        lib().oc_reset(ctypes.byref(self.spec.params()), _dp(self.bias), _dp(self.x_prev), _dp(self.z))
        self.key = True

    def step(self, x_t, force: bool | None = None):
        """Advance one frame.  Returns (score [n,ho,wo], block mask [n,nby,nbx])."""
        s = self.spec
        x_t = _f64(x_t)
        assert x_t.shape == self.x_prev.shape
        score = np.empty((s.n, s.ho, s.wo), np.float64)
        mask = np.empty((s.n, s.nby, s.nbx), np.uint8)
        f = self.key or self.dense_mode if force is None else force
        rc = lib().oc_step(ctypes.byref(s.params()), _dp(self.w), _dp(self.phi), self.phi_bias, _dp(x_t),
                           _dp(self.x_prev), _dp(self.z), int(f), _dp(score), mask.ctypes.data_as(_UP))
        if rc < 0:
            raise MemoryError("oracle step: allocation failed")
        self.key = False
        return score, mask

    def step_warped(self, x_t, flow, force: bool | None = None):
        """Advance one frame with a warped residual (Sec. 3.4, Eq. 10-11):
        r_t = x_t - T(x_{t-1}), z~_t = T~(z~_{t-1}) + g (.) (w * r_t), T and T~
        bilinear with the per-pixel flow [n, h, w, 2] = (dy, dx).  A key frame
        has no previous frame to warp: it is the plain key-frame step."""
        if self.key:
            return self.step(x_t, force)
        s = self.spec
        x_t = _f64(x_t)
        flow = _f64(flow)
        assert x_t.shape == self.x_prev.shape and flow.shape == (s.n, s.h, s.w, 2)
        score = np.empty((s.n, s.ho, s.wo), np.float64)
        mask = np.empty((s.n, s.nby, s.nbx), np.uint8)
        f = self.dense_mode if force is None else force
        rc = lib().oc_step_warped(ctypes.byref(s.params()), _dp(self.w), _dp(self.phi), self.phi_bias, _dp(x_t),
                                  _dp(self.x_prev), _dp(self.z), _dp(flow), int(f), _dp(score),
                                  mask.ctypes.data_as(_UP))
        if rc == -2:
            raise ValueError("warped residuals need a layer that keeps the frame size (stride 1, same padding)")
        if rc < 0:
            raise MemoryError("oracle step: allocation failed")
        return score, mask


def warp(x, flow):
    """T of Sec. 3.4: x [n, h, w, c] sampled at p + flow(p) by bilinear interpolation, zero outside."""
    x = _f64(x)
    flow = _f64(flow)
    n, h, w, c = x.shape
    out = np.empty_like(x)
    lib().oc_warp(n, h, w, c, _dp(flow), _dp(x), _dp(out))
    return out


class SampledOracleLayer:
    """The same recurrence with z kept only at chosen output locations.

    The gate is evaluated over the whole frame every step, so the sampled z
    values follow exactly the recurrence of the full state."""

    def __init__(self, spec: LayerSpec, w, samples_nij, bias=None, dense_mode: bool = False, phi=None,
                 phi_bias: float = 0.0):
        self.spec = spec
        self.w = _f64(w)
        self.phi = None if phi is None else _f64(phi)
        self.phi_bias = float(phi_bias)
        self.samples = np.ascontiguousarray(samples_nij, dtype=np.int32).reshape(-1, 3)
        self.bias = None if bias is None else _f64(bias)
        self.dense_mode = bool(dense_mode)
        self.x_prev = np.zeros((spec.n, spec.h, spec.w, spec.c_in), np.float64)
        self.z = np.zeros((len(self.samples), spec.c_out), np.float64)
        self.reset()

    def reset(self) -> None:
        self.x_prev[...] = 0.0
        self.z[...] = 0.0 if self.bias is None else self.bias[None, :]
        self.key = True

    def preset(self, x_prev, z_samples=None) -> None:
        """Start from a given state instead of a key frame (used for timing samples)."""
        self.x_prev[...] = _f64(x_prev)
        if z_samples is not None:
            self.z[...] = _f64(z_samples)
        self.key = False

    def step(self, x_t, force: bool | None = None):
        s = self.spec
        x_t = _f64(x_t)
        mask = np.empty((s.n, s.nby, s.nbx), np.uint8)
        f = self.key or self.dense_mode if force is None else force
        rc = lib().oc_step_sampled(ctypes.byref(s.params()), _dp(self.w), _dp(self.phi), self.phi_bias, _dp(x_t),
                                   _dp(self.x_prev), len(self.samples), self.samples.ctypes.data_as(_IP),
                                   _dp(self.z), int(f), mask.ctypes.data_as(_UP))
        if rc < 0:
            raise MemoryError("oracle step: allocation failed")
        self.key = False
        return mask
