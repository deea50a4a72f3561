"""Python binding of the Skip-Conv C ABI.

The ``skipconv_*`` functions mirror include/skipconv.h one to one and only
marshal arguments (device pointers as ints, or objects with ``data_ptr()``).
``SkipConvLayer`` wraps a handle with torch tensors for device memory and the
current CUDA stream; every step of the method runs in the library's kernels.
"""
from __future__ import annotations

import ctypes

from . import _lib
from ._lib import (ACT_NONE, ACT_RELU, ACT_SILU, BF16, F32, GATE_GUMBEL, GATE_INPUT_MEAN, GATE_INPUT_SUM,  # noqa: F401
                   GATE_OUTPUT, PATH_AUTO, PATH_CUDA_CORE, PATH_CUDA_CORE_SEPARATE, PATH_TENSOR_CORE,
                   PATH_TENSOR_CORE_SEPARATE, Info,
                   Params, SkipConvError, check)


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


# ------------------------------------------------------------- ABI mirror
def skipconv_create(params: Params, weights_oihw, bias=None, stream=None) -> int:
    h = ctypes.c_void_p()
    st = _lib.lib().skipconv_create(ctypes.byref(params), _ptr(weights_oihw), _ptr(bias),
                                    _ptr(stream) if stream is not None and not isinstance(stream, int) else stream,
                                    ctypes.byref(h))
    check("skipconv_create", st)
    return h.value


def skipconv_reset_state(handle: int) -> None:
    check("skipconv_reset_state", _lib.lib().skipconv_reset_state(handle))


def skipconv_step(handle: int, x_t, shortcut=None) -> None:
    check("skipconv_step", _lib.lib().skipconv_step(handle, _ptr(x_t), _ptr(shortcut)))


def skipconv_step_host(handle: int, x_t_host, z_out_host=None) -> None:
    check("skipconv_step_host", _lib.lib().skipconv_step_host(handle, _ptr(x_t_host), _ptr(z_out_host)))


def skipconv_step_host_async(handle: int, x_t_host, z_out_host=None) -> None:
    check("skipconv_step_host_async",
          _lib.lib().skipconv_step_host_async(handle, _ptr(x_t_host), _ptr(z_out_host)))


def skipconv_step_host_sparse_async(handle: int, x_t_host, z_blocks_host, list_host, count_host) -> None:
    check("skipconv_step_host_sparse_async",
          _lib.lib().skipconv_step_host_sparse_async(handle, _ptr(x_t_host), _ptr(z_blocks_host), _ptr(list_host),
                                                     _ptr(count_host)))


def skipconv_sync(handle: int) -> None:
    check("skipconv_sync", _lib.lib().skipconv_sync(handle))


def skipconv_destroy(handle: int) -> int:
    return _lib.lib().skipconv_destroy(handle)


def _get_ptr(fn: str, handle: int) -> int:
    p = ctypes.c_void_p()
    check(fn, getattr(_lib.lib(), fn)(handle, ctypes.byref(p)))
    return p.value or 0


def skipconv_get_z(handle: int) -> int:
    return _get_ptr("skipconv_get_z", handle)


def skipconv_get_y(handle: int) -> int:
    return _get_ptr("skipconv_get_y", handle)


def skipconv_get_prev_input(handle: int) -> int:
    return _get_ptr("skipconv_get_prev_input", handle)


def skipconv_get_gate(handle: int):
    m, l, c = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    check("skipconv_get_gate", _lib.lib().skipconv_get_gate(handle, ctypes.byref(m), ctypes.byref(l), ctypes.byref(c)))
    return m.value, l.value, c.value


def skipconv_gate_noalloc(params: Params, x_t, x_prev, block_mask, active_list, active_count, stream=None) -> None:
    check("skipconv_gate_noalloc", _lib.lib().skipconv_gate_noalloc(
        ctypes.byref(params), _ptr(x_t), _ptr(x_prev), _ptr(block_mask), _ptr(active_list), _ptr(active_count),
        _ptr(stream) if stream is not None and not isinstance(stream, int) else stream))


def skipconv_set_gate_weights(handle: int, phi_oihw, phi_bias: float = 0.0) -> None:
    check("skipconv_set_gate_weights", _lib.lib().skipconv_set_gate_weights(handle, _ptr(phi_oihw), float(phi_bias)))


def skipconv_step_warped(handle: int, x_t, flow, shortcut=None) -> None:
    """A step with a warped residual (Eq. 10-11); flow: float32 [n, h, w, 2] (dy, dx) on the device."""
    check("skipconv_step_warped", _lib.lib().skipconv_step_warped(handle, _ptr(x_t), _ptr(shortcut), _ptr(flow)))


def skipconv_link_inputs(handle: int, producer_x: int | None, producer_sc: int | None = None) -> None:
    """Stack propagation: this layer's x_t is producer_x's y (and its shortcut
    producer_sc's y); see include/skipconv.h.  producer_x = None unlinks."""
    check("skipconv_link_inputs", _lib.lib().skipconv_link_inputs(handle, producer_x, producer_sc))


def skipconv_get_info(handle: int) -> Info:
    info = Info()
    check("skipconv_get_info", _lib.lib().skipconv_get_info(handle, ctypes.byref(info)))
    return info


def skipconv_get_stats(handle: int):
    nb, nl, macs = ctypes.c_longlong(), ctypes.c_longlong(), ctypes.c_double()
    check("skipconv_get_stats", _lib.lib().skipconv_get_stats(handle, ctypes.byref(nb), ctypes.byref(nl),
                                                              ctypes.byref(macs)))
    return nb.value, nl.value, macs.value


def skipconv_check_device(handle: int) -> int:
    return _lib.lib().skipconv_check_device(handle)


def skipconv_selftest_timeout(handle: int, limit_ns: int) -> int:
    """Status of a kernel whose bounded wait runs out (SKIPCONV_ERR_TIMEOUT); the handle is then spent."""
    return _lib.lib().skipconv_selftest_timeout(handle, int(limit_ns))


def skipconv_profile(handle: int, enable: bool) -> None:
    check("skipconv_profile", _lib.lib().skipconv_profile(handle, int(bool(enable))))


def skipconv_profile_read(handle: int):
    """Returns (launches, ms), lists of PROFILE_KINDS per kernel kind: gate_pixel, gate_block, conv,
    y_refresh, fused tensor-core step, one-launch CUDA-core step, warp pass of a warped step."""
    launches = (ctypes.c_longlong * _lib.PROFILE_KINDS)()
    ms = (ctypes.c_double * _lib.PROFILE_KINDS)()
    check("skipconv_profile_read", _lib.lib().skipconv_profile_read(handle, launches, ms))
    return list(launches), list(ms)


# ------------------------------------------------------- torch convenience
class SkipConvLayer:
    """One Skip-Conv layer on the current CUDA device and stream.

    weights: OIHW tensor (float32 or bfloat16, the layer's dtype); bias: float32
    [c_out] or None.  Frames are NHWC tensors [n, h, w, c_in] of the same dtype.
    """

    def __init__(self, n_streams, c_in, c_out, h, w, k=3, stride=1, pad=1, groups=1, block=8, eps=0.05,
                 gate=GATE_INPUT_MEAN, dtype="bf16", activation=ACT_NONE, emit_y=False, dense_mode=False,
                 conv_path=PATH_AUTO, weights=None, bias=None, stream=None, key_interval=0, gate_weights=None,
                 gate_bias=0.0):
        import torch
        self.torch = torch
        self.dtype = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.params = Params(n_streams, c_in, c_out, h, w, k, k, stride, pad, groups, block, float(eps), gate,
                             BF16 if dtype == "bf16" else F32, activation, int(bool(emit_y)), int(bool(dense_mode)),
                             conv_path, int(key_interval))
        dev = torch.device("cuda", torch.cuda.current_device())
        w_t = torch.as_tensor(weights).to(device=dev, dtype=self.dtype).contiguous()
        b_t = None if bias is None else torch.as_tensor(bias).to(device=dev, dtype=torch.float32).contiguous()
        self.stream = stream if stream is not None else torch.cuda.current_stream(dev)
        self.handle = skipconv_create(self.params, w_t, b_t, self.stream.cuda_stream)
        if gate_weights is not None:        # Gumbel gate function phi [1, c_in, k, k] (or [c_in, k, k])
            phi = torch.as_tensor(gate_weights).to(device=dev, dtype=torch.float32).contiguous()
            skipconv_set_gate_weights(self.handle, phi, gate_bias)
        self.info = skipconv_get_info(self.handle)
        self.shape_in = (n_streams, h, w, c_in)
        self.shape_out = (n_streams, self.info.ho, self.info.wo, c_out)
        self.device = dev

    def close(self):
        if getattr(self, "handle", None):
            skipconv_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- copies of the library-owned state, for inspection (stream-ordered)
    def _view(self, ptr, shape, dtype):
        torch = self.torch
        cur = torch.cuda.current_stream(self.device)
        cur.wait_stream(self.stream)
        return device_tensor(ptr, shape, dtype).clone()

    def step(self, x_t, shortcut=None) -> None:
        assert tuple(x_t.shape) == self.shape_in and x_t.dtype == self.dtype and x_t.is_contiguous()
        if shortcut is not None:
            assert tuple(shortcut.shape) == self.shape_out and shortcut.dtype == self.dtype
        skipconv_step(self.handle, x_t, shortcut)

    def step_warped(self, x_t, flow, shortcut=None) -> None:
        """One step with a warped residual (Eq. 10-11): flow float32 [n, h, w, 2] = (dy, dx)."""
        assert tuple(x_t.shape) == self.shape_in and x_t.dtype == self.dtype and x_t.is_contiguous()
        n, h, w = self.shape_in[:3]
        assert tuple(flow.shape) == (n, h, w, 2) and flow.dtype == self.torch.float32 and flow.is_contiguous()
        skipconv_step_warped(self.handle, x_t, flow, shortcut)

    def reset(self) -> None:
        skipconv_reset_state(self.handle)

    def link(self, producer_x=None, producer_sc=None) -> None:
        """Stack propagation: x_t will be producer_x.y() (and the shortcut
        producer_sc.y()) at every step; None unlinks."""
        skipconv_link_inputs(self.handle, None if producer_x is None else producer_x.handle,
                             None if producer_sc is None else producer_sc.handle)

    def z(self):
        return self._view(skipconv_get_z(self.handle), self.shape_out, self.torch.float32)

    def y(self):
        p = skipconv_get_y(self.handle)
        return None if not p else self._view(p, self.shape_out, self.dtype)

    def prev_input(self):
        return self._view(skipconv_get_prev_input(self.handle), self.shape_in, self.dtype)

    def gate(self):
        """(block mask [n, nby, nbx] uint8, sorted open-block ids, count)."""
        torch = self.torch
        m, l, c = skipconv_get_gate(self.handle)
        n = self.shape_in[0] * self.info.nby * self.info.nbx
        mask = self._view(m, (self.shape_in[0], self.info.nby, self.info.nbx), torch.uint8)
        cnt = int(self._view(c, (1,), torch.int32).item())
        lst = self._view(l, (n,), torch.int32)[:cnt]
        return mask, torch.sort(lst).values, cnt

    def stats(self):
        return skipconv_get_stats(self.handle)


class _DeviceArray:
    """Minimal __cuda_array_interface__ exporter for a library-owned pointer."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(int(v) for v in shape), "typestr": typestr,
                                         "data": (int(ptr), False), "version": 2, "strides": None}


def device_tensor(ptr: int, shape, dtype):
    """Zero-copy torch view of device memory owned by the library."""
    import torch
    typestr = {torch.float32: "<f4", torch.bfloat16: "<i2", torch.uint8: "|u1", torch.int32: "<i4"}[dtype]
    t = torch.as_tensor(_DeviceArray(ptr, shape, typestr), device="cuda")
    return t.view(torch.bfloat16) if dtype == torch.bfloat16 else t
