"""Failure detection without a GPU fault: a kernel whose bounded wait is never
satisfied (a barrier that nothing completes) gives up after its limit and
records a timeout in the handle's device error word, the path every stuck
wait of the library's kernels takes.  The host then reads SKIPCONV_ERR_TIMEOUT,
the spent handle refuses work, and the context stays usable: a fresh handle
steps and matches the oracle."""
import numpy as np
import pytest
import torch

import synth
from harness import gpu_layer, to_device
from oracle import LayerSpec, OracleLayer
from paper_2104_11487_gb300 import skipconv_check_device, skipconv_selftest_timeout
from paper_2104_11487_gb300._lib import SKIPCONV_ERR_INVALID, SKIPCONV_ERR_TIMEOUT, SkipConvError

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_is_reported_and_the_context_survives():
    spec = LayerSpec(n=1, c_in=16, c_out=16, h=16, w=16, k=3, block=4, eps=0.05)
    rng = np.random.default_rng(5)
    w = synth.he_weights(rng, 16, 16, 3, bf16=True)
    spent = gpu_layer(spec, w, None, "bf16")
    x = to_device(synth.round_to_bf16(rng.standard_normal((1, 16, 16, 16)).astype(np.float32)), "bf16")
    try:
        assert skipconv_selftest_timeout(spent.handle, 0) == SKIPCONV_ERR_INVALID
        assert skipconv_selftest_timeout(spent.handle, 2_000_000) == SKIPCONV_ERR_TIMEOUT   # 2 ms
        assert skipconv_check_device(spent.handle) == SKIPCONV_ERR_TIMEOUT
        with pytest.raises(SkipConvError) as ei:
            spent.step(x)
        assert ei.value.status == SKIPCONV_ERR_TIMEOUT
    finally:
        spent.close()
    torch.cuda.synchronize()
    # a fresh handle in the same context works
    fresh = gpu_layer(spec, w, None, "bf16")
    try:
        ref = OracleLayer(spec, w, None)
        ref.step(x.float().cpu().numpy().astype(np.float64))
        fresh.step(x)
        z = fresh.z().cpu().numpy().astype(np.float64)
        rms = float(np.sqrt(np.mean(ref.z ** 2)))
        assert np.abs(z - ref.z).max() <= 2e-2 * rms
        assert skipconv_check_device(fresh.handle) == 0
    finally:
        fresh.close()
