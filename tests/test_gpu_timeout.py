"""Device-side timeouts reported as a status (no GPU fault involved).

The output-error contraction (also the clipping search's) hands work between its warps through
shared-memory barriers, and every wait is bounded.  With the test hook on, the kernel's tile-copy
thread issues no copies: every wait of the kernel runs out with nothing in flight (no copy issued,
no MMA issued), the kernel unwinds, the errors read NaN and mpq_device_status reports
MPQ_TIMEOUT_OUTPUT_ERROR (MPQ_TIMEOUT_CLIP for the clipping search).  The wait budget is set short
(a few ms) for the test and restored after it; the same context then computes correct results
again."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu

SHORT_WAIT = 1 << 22     # SM clocks, about 2 ms


def _layer(gpu, oracle, C=40, d=128, N=300, K=3):
    W = wlm.random_weights(C, d, 77, "normal")
    q = oracle.quantize_layer(W, 4, 16, K)
    X = wlm.random_calibration(N, d, 78)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    return (X, W, q), (t(X), t(W), t(q["codes"]), t(q["scales"]), K)


def test_withheld_copies_time_out_and_are_reported(gpu, oracle):
    (X, W, q), args = _layer(gpu, oracle)
    assert binding.mpq_device_status() == 0            # nothing recorded before
    try:
        binding.mpq_set_wait_limit(SHORT_WAIT)
        binding.mpq_test_withhold_copies(True)
        err = binding.mpq_output_error(*args)
        flags = binding.mpq_device_status()
    finally:
        binding.mpq_test_withhold_copies(False)
        binding.mpq_set_wait_limit(0)
    assert flags & binding.MPQ_TIMEOUT_OUTPUT_ERROR
    assert not flags & binding.MPQ_TIMEOUT_DRAIN       # nothing was in flight to drain
    assert torch.isnan(err).all()
    assert binding.mpq_device_status() == 0            # taking the word cleared it
    # the context is still usable: the same call is correct again
    good = binding.mpq_output_error(*args)
    assert binding.mpq_device_status() == 0
    err_or = oracle.output_error(X, 1, W, q["codes"], q["scales"], args[-1])
    g = good.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(g - err_or) / np.abs(err_or)) <= 1e-5


def test_clip_search_withheld_copies(gpu, oracle):
    """The clipping search's contraction (A tiles copied from the residual planes, a relay warp
    per CTA) unwinds the same way: every error NaN, no factor chosen, MPQ_TIMEOUT_CLIP reported,
    nothing left to drain; then the same call is correct."""
    W = wlm.random_weights(30, 128, 79, "laplace")
    X = wlm.random_calibration(300, 128, 80)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    mode = binding.MPQ_CLIP_PER_CHANNEL
    assert binding.mpq_device_status() == 0
    try:
        binding.mpq_set_wait_limit(SHORT_WAIT)
        binding.mpq_test_withhold_copies(True)
        clip, err, best = binding.mpq_clip_search(t(X), t(W), 4, 20, mode)
        flags = binding.mpq_device_status()
    finally:
        binding.mpq_test_withhold_copies(False)
        binding.mpq_set_wait_limit(0)
    assert flags & binding.MPQ_TIMEOUT_CLIP
    assert not flags & binding.MPQ_TIMEOUT_DRAIN
    assert torch.isnan(err).all() and bool((best == -1).all())
    assert binding.mpq_device_status() == 0
    clip, err, best = binding.mpq_clip_search(t(X), t(W), 4, 20, mode)
    assert binding.mpq_device_status() == 0
    o_clip = oracle.clip_candidates(W, 20, mode)
    o_err = oracle.clip_errors(X, 1, W, 4, o_clip)
    e = err.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(e - o_err) / np.abs(o_err)) <= 1e-5


def test_status_through_the_c_abi(gpu):
    lib = binding.load()
    import ctypes
    flags = ctypes.c_uint(123)
    assert lib.mpq_device_status(None, ctypes.byref(flags)) == 0
    assert flags.value == 0
    assert lib.mpq_device_status(None, None) == 0
