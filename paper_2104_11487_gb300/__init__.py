"""GB300 (sm_103a) Skip-Convolution layer step (arXiv 2104.11487).

The compute lives in libskipconv.so (CUDA, C ABI in include/skipconv.h);
this package builds it and binds it.  There is no CPU fallback: importing a
binding whose library cannot be built or loaded raises.
"""
from ._build import build_library  # noqa: F401
from .skipconv import (SkipConvLayer, device_tensor, skipconv_check_device, skipconv_create,  # noqa: F401
                       skipconv_destroy, skipconv_gate_noalloc, skipconv_get_gate, skipconv_get_info,
                       skipconv_get_prev_input,
                       skipconv_get_stats, skipconv_get_y, skipconv_get_z, skipconv_profile, skipconv_profile_read,
                       skipconv_link_inputs, skipconv_reset_state, skipconv_selftest_timeout,
                       skipconv_set_gate_weights, skipconv_step,
                       skipconv_step_host, skipconv_step_host_async, skipconv_step_host_sparse_async,
                       skipconv_step_warped, skipconv_sync)
