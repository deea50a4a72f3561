"""The C-ABI library builds, loads without a GPU and exports every symbol
that include/skipconv.h declares; argument validation is host-side."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "skipconv.h")


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"SKIPCONV_API\s+[\w\s\*]+?\b(skipconv_\w+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    for required in ("skipconv_create", "skipconv_reset_state", "skipconv_step", "skipconv_destroy"):
        assert required in names
    assert len(names) >= 14


def test_library_exports_every_declared_symbol():
    from paper_2104_11487_gb300 import _lib
    L = _lib.lib()
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing
    # the ctypes table covers the header exactly
    assert set(_lib.SIGNATURES) == set(declared_functions())


def test_exported_symbols_are_only_the_abi():
    import subprocess
    from paper_2104_11487_gb300 import _lib
    _lib.lib()
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.library_path()], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("nm unavailable")
    syms = [l.split()[-1] for l in out.stdout.splitlines() if l.strip()]
    ours = [s for s in syms if s.startswith("skipconv_")]
    assert sorted(ours) == declared_functions()


def test_params_struct_layout():
    from paper_2104_11487_gb300 import _lib
    # 11 ints, 1 float, 6 ints, no padding
    assert ctypes.sizeof(_lib.Params) == 19 * 4
    assert _lib.Params.eps.offset == 11 * 4


def test_status_strings():
    from paper_2104_11487_gb300 import _lib
    L = _lib.lib()
    assert L.skipconv_status_string(0) == b"SKIPCONV_OK"
    assert L.skipconv_status_string(-6) == b"SKIPCONV_ERR_DEVICE"
    assert L.skipconv_status_string(42) == b"SKIPCONV_UNKNOWN_STATUS"


def test_host_side_validation_without_gpu():
    """Invalid arguments are rejected before any CUDA call."""
    from paper_2104_11487_gb300 import _lib
    L = _lib.lib()
    h = ctypes.c_void_p()
    assert L.skipconv_create(None, None, None, None, ctypes.byref(h)) == _lib.SKIPCONV_ERR_INVALID
    p = _lib.Params(1, 4, 4, 8, 8, 3, 3, 1, 1, 1, 8, 0.05, 0, 1, 0, 0, 0, 0)
    p.c_in = 0
    assert L.skipconv_create(ctypes.byref(p), ctypes.c_void_p(16), None, None, ctypes.byref(h)) == \
        _lib.SKIPCONV_ERR_INVALID
    p.c_in, p.groups = 4, 3
    assert L.skipconv_create(ctypes.byref(p), ctypes.c_void_p(16), None, None, ctypes.byref(h)) == \
        _lib.SKIPCONV_ERR_INVALID
    assert b"groups" in L.skipconv_last_error()
    p.groups, p.eps = 1, -1.0
    assert L.skipconv_create(ctypes.byref(p), ctypes.c_void_p(16), None, None, ctypes.byref(h)) == \
        _lib.SKIPCONV_ERR_INVALID
    p.eps, p.dtype = 0.05, 7
    assert L.skipconv_create(ctypes.byref(p), ctypes.c_void_p(16), None, None, ctypes.byref(h)) == \
        _lib.SKIPCONV_ERR_INVALID
    assert h.value is None
    # NULL handles
    assert L.skipconv_step(None, None, None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_reset_state(None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_step_host(None, None, None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_step_host_async(None, None, None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_sync(None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_step_warped(None, None, None, None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_link_inputs(None, None, None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_selftest_timeout(None, 1000) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_check_device(None) == _lib.SKIPCONV_ERR_INVALID
    assert L.skipconv_destroy(None) == _lib.SKIPCONV_OK


def test_oracle_and_library_share_no_code():
    """The oracle is independent of the CUDA path: neither side includes or
    imports the other."""
    import glob
    for f in glob.glob(os.path.join(ROOT, "oracle", "*")):
        if os.path.isfile(f) and f.endswith((".py", ".c", ".h")):
            text = open(f).read()
            assert "paper_2104_11487_gb300" not in text.replace("never imports it", "").replace(
                "(``paper_2104_11487_gb300``)", "")
            assert "skipconv.h" not in text
    for f in glob.glob(os.path.join(ROOT, "paper_2104_11487_gb300", "**", "*.*"), recursive=True):
        if f.endswith((".py", ".cu", ".h", ".cuh")) and "_build" not in f:
            text = open(f).read()
            assert "import oracle" not in text and "from oracle" not in text and "skipconv_oracle" not in text
