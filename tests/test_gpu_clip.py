"""Parity of mpq_clip_search (Eq. 12, output-error-driven clipping factor) with the oracle, through
the C ABI: candidate factors bit-exact, errors within the output-error bar, and both argmins
bit-exact given the device's fp32 error table."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm
from _parity import compare_err

pytestmark = pytest.mark.gpu

MODES = (binding.MPQ_CLIP_PER_CHANNEL, binding.MPQ_CLIP_PER_LAYER)


def run_both(oracle, X, W, bits, n_cand, mode, groups=1):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to("cuda:0")
    clip, err, best = binding.mpq_clip_search(t(X), t(W), bits, n_cand, mode, groups=groups)
    torch.cuda.synchronize()
    clip, err, best = clip.cpu().numpy(), err.cpu().numpy(), best.cpu().numpy()
    o_clip = oracle.clip_candidates(W, n_cand, mode)
    assert np.array_equal(clip, o_clip, equal_nan=True)
    o_err = oracle.clip_errors(X, groups, W, bits, o_clip, threads=8)
    compare_err(err, o_err)
    assert np.array_equal(best, oracle.clip_select(err, mode))
    return clip, err, best, o_err


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("C,d,N,n_cand", [
    # d % 16 == 0: CTA-pair tensor-core path -- several pair tiles, a part-filled odd CTA, ragged
    # row tiles split over clusters, 1 to 32 candidates
    (50, 256, 600, 20), (13, 64, 100, 32), (130, 128, 300, 7), (3, 48, 20, 1), (64, 576, 512, 20),
    # other rows: shared-memory path
    (11, 147, 129, 20), (4, 33, 70, 5), (2, 17, 300, 32),
])
def test_shared_input(gpu, oracle, mode, C, d, N, n_cand):
    W = wlm.random_weights(C, d, 100 + C + d, "laplace")
    X = wlm.random_calibration(N, d, 200 + N)
    run_both(oracle, X, W, 4, n_cand, mode)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("C,d,N,n_cand", [(6, 9, 100, 20), (40, 9, 1024, 20), (3, 25, 77, 8)])
def test_per_channel_input(gpu, oracle, mode, C, d, N, n_cand):
    W = wlm.random_weights(C, d, 300 + C, "laplace")
    X = wlm.random_calibration(N, d, 17, groups=C)
    run_both(oracle, X, W, 4, n_cand, mode, groups=C)


@pytest.mark.parametrize("bits", [2, 3, 8])
def test_bit_widths(gpu, oracle, bits):
    W = wlm.random_weights(20, 96, 7 + bits, "normal")
    X = wlm.random_calibration(64, 96, 9)
    run_both(oracle, X, W, bits, 20, binding.MPQ_CLIP_PER_CHANNEL)


def test_heavy_tail_prefers_clipping(gpu, oracle):
    """A few outlier weights: the output error prefers K < max|w| for most channels."""
    rng = np.random.default_rng(5)
    W = (rng.standard_normal((32, 256)) * 0.02).astype(np.float32)
    W[np.arange(32), rng.integers(0, 256, 32)] *= 30
    X = wlm.random_calibration(300, 256, 3)
    _, _, best, _ = run_both(oracle, X, W, 4, 20, binding.MPQ_CLIP_PER_CHANNEL)
    assert np.mean(best < 19) > 0.5


def test_config1_layer(gpu, oracle):
    wl = wlm.WORKLOADS["c1"]
    W = wlm.make_weights(wl, 0)
    X = wlm.make_calibration(wl, 0)
    for mode in MODES:
        run_both(oracle, X, W, 4, 20, mode)


def test_nonfinite_and_zero_channels(gpu, oracle):
    W = wlm.random_weights(6, 64, 3, "normal")
    W[1, 5] = np.nan
    W[4, :] = 0.0
    X = wlm.random_calibration(40, 64, 4)
    clip, err, best, _ = run_both(oracle, X, W, 4, 20, binding.MPQ_CLIP_PER_CHANNEL)
    assert best[1] == -1 and np.all(np.isnan(err[1]))
    assert best[4] == 0 and np.all(err[4] == 0)
    _, err, best, _ = run_both(oracle, X, W, 4, 20, binding.MPQ_CLIP_PER_LAYER)
    assert np.all(best == -1) and np.all(np.isnan(err))


def test_per_layer_small_channels(gpu, oracle):
    """One K for the layer while some channels are orders of magnitude smaller: their candidates
    quantize everything to 0, so their residuals are the weights themselves, far below s/2; the
    operand scale follows their own max|w| and the errors keep the 1e-5 bar."""
    W = wlm.random_weights(24, 256, 41, "laplace")
    W[3] *= np.float32(1e-4)
    W[7] *= np.float32(1e-9)
    W[11] *= np.float32(1e-6)
    X = wlm.random_calibration(300, 256, 42)
    run_both(oracle, X, W, 4, 20, binding.MPQ_CLIP_PER_LAYER)
    run_both(oracle, X, W, 4, 20, binding.MPQ_CLIP_PER_CHANNEL)


def test_full_size_sampled(gpu, oracle):
    """c5's up_proj shape (11008 x 4096, N = 2048) in the launch the bench times, checked on
    sampled channels against the oracle; per-layer argmin recomputed from the device table."""
    wl = wlm.WORKLOADS["c5"]
    W = wlm.make_weights(wl, 1)
    X = wlm.make_calibration(wl, 1)
    t = lambda a: torch.from_numpy(a).to("cuda:0")
    for mode in MODES:
        clip, err, best = binding.mpq_clip_search(t(X), t(W), 4, 20, mode)
        torch.cuda.synchronize()
        clip, err, best = clip.cpu().numpy(), err.cpu().numpy(), best.cpu().numpy()
        o_clip = oracle.clip_candidates(W, 20, mode)
        assert np.array_equal(clip, o_clip)
        for c0 in (0, 5000, 11008 - 8):
            o_err = oracle.clip_errors(X, 1, W, 4, o_clip, channels=(c0, c0 + 8), threads=8)
            compare_err(err[c0:c0 + 8], o_err[c0:c0 + 8])
        assert np.array_equal(best, oracle.clip_select(err, mode))


def test_planes_in_chunks(gpu, oracle):
    """Residual planes over 4 GiB (4100 channels x 32 candidates x d = 8192 x 4 bytes) are written
    and contracted in two chunks of whole channels; channels on both sides of the boundary (4096)
    against the oracle."""
    C, d, N, nc = 4100, 8192, 256, 32
    W = wlm.random_weights(C, d, 91, "laplace")
    X = wlm.random_calibration(N, d, 92)
    t = lambda a: torch.from_numpy(a).to("cuda:0")
    clip, err, best = binding.mpq_clip_search(t(X), t(W), 4, nc, binding.MPQ_CLIP_PER_CHANNEL)
    torch.cuda.synchronize()
    clip, err, best = clip.cpu().numpy(), err.cpu().numpy(), best.cpu().numpy()
    o_clip = oracle.clip_candidates(W, nc, binding.MPQ_CLIP_PER_CHANNEL)
    assert np.array_equal(clip, o_clip)
    for c0 in (0, 4090, C - 4):
        o_err = oracle.clip_errors(X, 1, W, 4, o_clip, channels=(c0, c0 + 4), threads=8)
        compare_err(err[c0:c0 + 4], o_err[c0:c0 + 4])
    assert np.array_equal(best, oracle.clip_select(err, binding.MPQ_CLIP_PER_CHANNEL))

