"""The adaptive grid of Eq. 10 (Definition 1) through the C ABI against the oracle: grid sizes,
scales, codes and residual norms bit-exact per step, near ties of the objective allowed and
counted (tests/_parity.compare_adaptive).  Short channels against the oracle's plain enumeration
of the grid; long ones (grids of 1e9..1e10 points a step) against its piecewise search, which is
pinned to the enumeration in tests/test_oracle_pins.py."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm
from _parity import compare_adaptive

pytestmark = pytest.mark.gpu

BIG = 10 ** 15    # no refusal: the GPU search does not enumerate the grid


def run(W, bits, k_max, max_cand=BIG, dev="cuda:0"):
    codes, scales, rs, nc = binding.mpq_quantize_layer_adaptive(
        torch.from_numpy(np.ascontiguousarray(W)).to(dev), bits, k_max, max_cand=max_cand)
    torch.cuda.synchronize()
    return dict(codes=codes.cpu().numpy(), scales=scales.cpu().numpy(),
                resid_sq=rs.cpu().numpy(), ncand=nc.cpu().numpy())


def check(oracle, W, bits, k_max, cap=10 ** 7, piecewise=False, sample=None):
    """Both sides with the same candidate cap; a refused step is marked alike on both."""
    g = run(W, bits, k_max, max_cand=cap)
    Wo = W if sample is None else W[sample]
    o = oracle.quantize_adaptive(Wo, bits, k_max, max_candidates=cap, refuse="mark",
                                 piecewise=piecewise)
    if sample is not None:
        g = dict(codes=g["codes"][:, sample], scales=g["scales"][sample],
                 resid_sq=g["resid_sq"][sample], ncand=g["ncand"][sample])
    return compare_adaptive(g, o, bits, oracle)


@pytest.mark.parametrize("C,d,bits,k_max,dist,scale", [
    (64, 9, 4, 8, "laplace", 1.0),        # depthwise 3x3 filters
    (20, 1, 4, 3, "normal", 1.0),         # one weight: one distinct magnitude, gamma = eta
    (30, 2, 2, 4, "normal", 1.0),
    (16, 16, 3, 5, "t", 1.0),
    (8, 12, 6, 3, "normal", 0.01),        # 6-bit codes, small weights
    (4, 64, 4, 1, "normal", 1.0),
])
def test_adaptive_parity_enumerated(gpu, oracle, C, d, bits, k_max, dist, scale):
    W = (wlm.random_weights(C, d, 3 * C + d + bits, dist) * np.float32(scale)).astype(np.float32)
    check(oracle, W, bits, k_max)


@pytest.mark.parametrize("C,d,bits,k_max,dist", [
    (6, 147, 4, 3, "normal"),             # a first convolution's row, ragged length
    (5, 300, 2, 4, "t"),                  # b = 2: Q = {-1, 0, 1}
    (4, 256, 5, 2, "laplace"),
    (3, 1000, 3, 3, "normal"),
])
def test_adaptive_parity_long(gpu, oracle, C, d, bits, k_max, dist):
    W = wlm.random_weights(C, d, 11 * C + d, dist)
    check(oracle, W, bits, k_max, cap=BIG, piecewise=True)


def test_adaptive_repeated_magnitudes(gpu, oracle):
    """Repeated and sign-flipped magnitudes, zeros, an all-zero channel (null points)."""
    rng = np.random.default_rng(5)
    W = (np.round(rng.standard_normal((24, 9)) * 4) / 4).astype(np.float32)
    W[3] = 0.0
    W[4] = [0.5, -0.5] * 4 + [0.5]
    check(oracle, W, 4, 5)


def test_adaptive_depthwise_layer(gpu, oracle):
    """The MobileNetV2 set's largest depthwise layer (960 channels of 9 weights), eight points, on
    the GPU; its first 48 channels against the oracle's enumeration (grids up to 2e7 a step)."""
    wl = wlm.WORKLOADS["c4"]
    li = max((i for i, l in enumerate(wl.layers) if l.d == 9), key=lambda i: wl.layers[i].C)
    W = wlm.make_weights(wl, li)
    check(oracle, W, 4, wl.k_max, cap=10 ** 8, sample=np.arange(48))


def test_adaptive_resnet18_layer(gpu, oracle):
    """c2's 64 x 576 convolution (grids of ~1.5e9 points a step), all 64 channels on the GPU, 8
    of them against the oracle's piecewise search, four points."""
    wl = wlm.WORKLOADS["c2"]
    W = wlm.make_weights(wl, 1)
    check(oracle, W, 4, 4, cap=BIG, piecewise=True, sample=np.arange(0, 64, 8))


def test_adaptive_large_linear_channels(gpu, oracle):
    """Three channels of c5's 4096 x 4096 layer (N(0, 0.02^2) with outliers), eight points."""
    wl = wlm.WORKLOADS["c5"]
    W = wlm.make_weights(wl, 0, rows=(0, 3))
    check(oracle, W, 4, 8, cap=BIG, piecewise=True)


def test_adaptive_refused_and_nonfinite(gpu, oracle):
    W = wlm.random_weights(6, 9, 8, "normal")
    W[2, 4] = np.nan
    g = run(W, 4, 3, max_cand=10)                           # every grid is larger than 10
    nc, scales, codes, rs = g["ncand"], g["scales"], g["codes"], g["resid_sq"]
    assert np.all(nc[[0, 1, 3, 4, 5], 0] == -1) and np.all(nc[:, 1:] == 0) and np.all(nc[2] == 0)
    assert np.all(np.isnan(scales)) and np.all(codes == 0)
    assert np.all(np.isnan(rs[:, 1:])) and np.isnan(rs[2, 0])
    g = run(W, 4, 3, max_cand=10 ** 8)
    assert np.all(np.isnan(g["scales"][2])) and np.all(g["codes"][:, 2] == 0)
    keep = [0, 1, 3, 4, 5]
    o = oracle.quantize_adaptive(W[keep], 4, 3, max_candidates=10 ** 8, refuse="mark")
    sub = dict(codes=g["codes"][:, keep], scales=g["scales"][keep], resid_sq=g["resid_sq"][keep],
               ncand=g["ncand"][keep])
    compare_adaptive(sub, o, 4, oracle)


def test_adaptive_tiny_gap_zero_scales(gpu, oracle):
    """Subnormal weights: the minimal gap is a few 2^-149, so gamma is below the fp32 range and
    the grid's first scales fl(m gamma / Qmax) are 0 (codes 0, the objective ||r||^2) before
    the positive ones -- a case the definition decides among scale 0 and positive scales."""
    rng = np.random.default_rng(7)
    ints = rng.integers(-60, 61, size=(6, 12)).astype(np.float64)
    ints[0, :2] = [37, 38]                     # neighbouring magnitudes: the smallest gap
    W = (ints * 2.0 ** -149).astype(np.float32)
    assert np.all(np.abs(W[W != 0]) < np.finfo(np.float32).tiny)
    for bits in (2, 4):
        o = oracle.quantize_adaptive(W, bits, 3, max_candidates=10 ** 7, refuse="mark")
        assert np.any(np.float32(o["gamma"][:, 0] / (2 ** (bits - 1) - 1)) == 0.0)
        g = run(W, bits, 3, max_cand=10 ** 7)
        compare_adaptive(g, o, bits, oracle)
