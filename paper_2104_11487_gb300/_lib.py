"""ctypes view of libskipconv.so (include/skipconv.h).  Marshalling only."""
from __future__ import annotations

import ctypes
import os

from . import _build

c_int, c_void_p, c_float, c_longlong = ctypes.c_int, ctypes.c_void_p, ctypes.c_float, ctypes.c_longlong

SKIPCONV_OK = 0
SKIPCONV_ERR_INVALID = -1
SKIPCONV_ERR_UNSUPPORTED = -2
SKIPCONV_ERR_CUDA = -3
SKIPCONV_ERR_OOM = -4
SKIPCONV_ERR_TIMEOUT = -5
SKIPCONV_ERR_DEVICE = -6

GATE_INPUT_MEAN, GATE_INPUT_SUM, GATE_OUTPUT, GATE_GUMBEL = 0, 1, 2, 3
F32, BF16 = 0, 1
ACT_NONE, ACT_RELU, ACT_SILU = 0, 1, 2
PATH_AUTO, PATH_CUDA_CORE, PATH_TENSOR_CORE, PATH_TENSOR_CORE_SEPARATE, PATH_CUDA_CORE_SEPARATE = 0, 1, 2, 3, 4
PROFILE_KINDS = 7   # gate_pixel, gate_block, conv, y_refresh, fused tensor-core step, CUDA-core step, warp pass

# Every function the header declares, with its ctypes signature.
SIGNATURES = {
    "skipconv_create": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_reset_state": (c_int, [c_void_p]),
    "skipconv_step": (c_int, [c_void_p, c_void_p, c_void_p]),
    "skipconv_step_host": (c_int, [c_void_p, c_void_p, c_void_p]),
    "skipconv_step_host_async": (c_int, [c_void_p, c_void_p, c_void_p]),
    "skipconv_step_host_sparse_async": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_sync": (c_int, [c_void_p]),
    "skipconv_destroy": (c_int, [c_void_p]),
    "skipconv_get_z": (c_int, [c_void_p, c_void_p]),
    "skipconv_get_y": (c_int, [c_void_p, c_void_p]),
    "skipconv_get_prev_input": (c_int, [c_void_p, c_void_p]),
    "skipconv_get_gate": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_get_info": (c_int, [c_void_p, c_void_p]),
    "skipconv_get_stats": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_check_device": (c_int, [c_void_p]),
    "skipconv_selftest_timeout": (c_int, [c_void_p, c_longlong]),
    "skipconv_profile": (c_int, [c_void_p, c_int]),
    "skipconv_profile_read": (c_int, [c_void_p, c_void_p, c_void_p]),
    "skipconv_gate_noalloc": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_set_gate_weights": (c_int, [c_void_p, c_void_p, c_float]),
    "skipconv_link_inputs": (c_int, [c_void_p, c_void_p, c_void_p]),
    "skipconv_step_warped": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "skipconv_status_string": (ctypes.c_char_p, [c_int]),
    "skipconv_last_error": (ctypes.c_char_p, []),
}


class Params(ctypes.Structure):
    _fields_ = [(n, c_int) for n in ("n_streams", "c_in", "c_out", "h", "w", "k_h", "k_w", "stride", "pad",
                                     "groups", "block")] + [("eps", c_float)] + [
        (n, c_int) for n in ("gate", "dtype", "activation", "emit_y", "dense_mode", "conv_path", "key_interval")]


class Info(ctypes.Structure):
    _fields_ = [(n, c_int) for n in ("ho", "wo", "nby", "nbx", "conv_path", "num_sms")] + [
        ("state_bytes", ctypes.c_size_t), ("fused", c_int)]


class SkipConvError(RuntimeError):
    def __init__(self, fn: str, status: int, detail: str):
        super().__init__("%s failed: %s (%s)" % (fn, _status_name(status), detail))
        self.status = status


_lib = None


def _status_name(s: int) -> str:
    try:
        return lib().skipconv_status_string(s).decode()
    except Exception:
        return str(s)


def library_path() -> str:
    return _build.LIB


def lib(build: bool = True):
    """Load libskipconv.so (building it first if it is missing).  Raises if
    the CUDA library cannot be built or loaded: there is no fallback."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if build or not os.path.exists(path):
            path = _build.build_library()
        if not os.path.exists(path):
            raise RuntimeError("libskipconv.so is missing and could not be built")
        L = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def check(fn: str, status: int) -> None:
    if status != SKIPCONV_OK:
        raise SkipConvError(fn, status, lib().skipconv_last_error().decode(errors="replace"))
