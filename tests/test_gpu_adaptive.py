"""The adaptive grid of Eq. 10 (Definition 1) through the C ABI: codes, scales, residual norms and
each step's grid size bit-exact against the oracle's enumeration, on short channels."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu


def run(W, bits, k_max, max_cand=10 ** 7, dev="cuda:0"):
    codes, scales, rs, nc = binding.mpq_quantize_layer_adaptive(
        torch.from_numpy(np.ascontiguousarray(W)).to(dev), bits, k_max, max_cand=max_cand)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), scales.cpu().numpy(), rs.cpu().numpy(), nc.cpu().numpy()


def check(oracle, W, bits, k_max, cap=10 ** 7):
    """Both sides with the same candidate cap; a refused step is marked alike on both."""
    codes, scales, rs, nc = run(W, bits, k_max, max_cand=cap)
    o = oracle.quantize_adaptive(W, bits, k_max, max_candidates=cap, refuse="mark")
    np.testing.assert_array_equal(codes, o["codes"])
    np.testing.assert_array_equal(scales, o["scales"])
    np.testing.assert_array_equal(rs, o["resid_sq"].astype(np.float32))
    np.testing.assert_array_equal(nc, o["ncand"])


@pytest.mark.parametrize("C,d,bits,k_max,dist,scale", [
    (64, 9, 4, 8, "laplace", 1.0),        # depthwise 3x3 filters
    (20, 1, 4, 3, "normal", 1.0),         # one weight: one distinct magnitude, gamma = eta
    (30, 2, 2, 4, "normal", 1.0),
    (16, 16, 3, 5, "t", 1.0),
    (8, 12, 6, 3, "normal", 0.01),        # 6-bit codes, small weights
    (4, 64, 4, 1, "normal", 1.0),         # the longest channel taken
])
def test_adaptive_parity(gpu, oracle, C, d, bits, k_max, dist, scale):
    W = (wlm.random_weights(C, d, 3 * C + d + bits, dist) * np.float32(scale)).astype(np.float32)
    check(oracle, W, bits, k_max)


def test_adaptive_repeated_magnitudes(gpu, oracle):
    """Repeated and sign-flipped magnitudes, zeros, an all-zero channel (null points)."""
    rng = np.random.default_rng(5)
    W = (np.round(rng.standard_normal((24, 9)) * 4) / 4).astype(np.float32)
    W[3] = 0.0
    W[4] = [0.5, -0.5] * 4 + [0.5]
    check(oracle, W, 4, 5)


def test_adaptive_depthwise_layer(gpu, oracle):
    """The MobileNetV2 set's largest depthwise layer (960 channels of 9 weights), eight points, on
    the GPU; its first 48 channels against the oracle (grids of up to 2e7 candidates a step)."""
    wl = wlm.WORKLOADS["c4"]
    li = max((i for i, l in enumerate(wl.layers) if l.d == 9), key=lambda i: wl.layers[i].C)
    W = wlm.make_weights(wl, li)
    codes, scales, rs, nc = run(W, 4, wl.k_max, max_cand=10 ** 8)
    o = oracle.quantize_adaptive(W[:48], 4, wl.k_max, max_candidates=10 ** 8, refuse="mark")
    np.testing.assert_array_equal(codes[:, :48], o["codes"])
    np.testing.assert_array_equal(scales[:48], o["scales"])
    np.testing.assert_array_equal(rs[:48], o["resid_sq"].astype(np.float32))
    np.testing.assert_array_equal(nc[:48], o["ncand"])


def test_adaptive_refused_and_nonfinite(gpu, oracle):
    W = wlm.random_weights(6, 9, 8, "normal")
    W[2, 4] = np.nan
    codes, scales, rs, nc = run(W, 4, 3, max_cand=10)        # every grid is larger than 10
    assert np.all(nc[[0, 1, 3, 4, 5], 0] == -1) and np.all(nc[:, 1:] == 0) and np.all(nc[2] == 0)
    assert np.all(np.isnan(scales)) and np.all(codes == 0)
    assert np.all(np.isnan(rs[:, 1:])) and np.isnan(rs[2, 0])
    codes, scales, rs, nc = run(W, 4, 3)
    assert np.all(np.isnan(scales[2])) and np.all(codes[:, 2] == 0)
    keep = [0, 1, 3, 4, 5]
    o = oracle.quantize_adaptive(W[keep], 4, 3, refuse="mark")
    np.testing.assert_array_equal(scales[keep], o["scales"])
    np.testing.assert_array_equal(codes[:, keep], o["codes"])
