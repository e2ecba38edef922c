"""Parity of mpq_quantize_layer (Algorithm 1, Eq. 7-9) with the oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm
from _parity import compare_quantize

pytestmark = pytest.mark.gpu


def run_gpu(W, bits, G, k_max, grid_frac=None, dev="cuda:0"):
    Wd = torch.from_numpy(W).to(dev)
    C, d = W.shape
    res = torch.empty((k_max, C, d), dtype=torch.float32, device=dev)
    codes, scales, rs, res = binding.mpq_quantize_layer(Wd, bits, G, k_max, grid_frac=grid_frac,
                                                        residuals=res)
    torch.cuda.synchronize()
    return dict(codes=codes.cpu().numpy(), scales=scales.cpu().numpy(),
                resid_sq=rs.cpu().numpy(), residuals=res.cpu().numpy())


def check(oracle, W, bits, G, k_max, grid_frac=None):
    gpu = run_gpu(W, bits, G, k_max, grid_frac)
    orc = oracle.quantize_layer(W, bits, G, k_max, grid_frac=grid_frac)
    return compare_quantize(W, gpu, orc, bits, G, k_max, grid_frac, oracle=oracle)


@pytest.mark.parametrize("C,d", [(1, 1), (3, 2), (2, 3), (5, 4), (7, 9), (4, 31), (6, 33),
                                 (64, 147), (9, 255), (64, 576), (3, 1000), (5, 1153)])
def test_shapes(gpu, oracle, C, d):
    W = wlm.random_weights(C, d, 1000 + C * 7 + d, "normal")
    rep = check(oracle, W, 4, 64, 4)
    assert rep["near_ties"] <= max(1, C * 4 // 50)


@pytest.mark.parametrize("C,d,bits,G,k_max,dist", [
    (960, 9, 4, 64, 8, "laplace"),      # the MobileNetV2 set's largest depthwise layer
    (50, 25, 3, 128, 6, "t"),
    (20, 32, 8, 256, 4, "normal"),      # the longest direct row, 8-bit codes (Qmax = 127)
    (30, 16, 2, 1024, 3, "normal"),     # the largest grid, b = 2
    (40, 1, 4, 7, 16, "normal"),        # one weight per channel, 16 points
])
def test_short_rows_direct(gpu, oracle, C, d, bits, G, k_max, dist):
    """Rows of at most 32 weights evaluate every candidate's P and N directly from the codes
    instead of through the lattice; the chosen scales, codes and residuals stay the definition's."""
    W = wlm.random_weights(C, d, 7 * C + d + G, dist)
    rep = check(oracle, W, bits, G, k_max)
    assert rep["near_ties"] <= max(1, C * k_max // 50)


def test_short_rows_custom_grid(gpu, oracle):
    W = wlm.random_weights(64, 9, 12, "laplace")
    gf = np.sort(np.random.default_rng(2).uniform(0.02, 1.0, 33)).astype(np.float32)
    check(oracle, W, 4, gf.size, 8, grid_frac=gf)


def test_max_dim(gpu, oracle):
    """The longest channel the library takes (d = 8192): residual, bins and lattice on chip."""
    W = wlm.random_weights(3, 8192, 81, "normal")
    rep = check(oracle, W, 4, 128, 4)
    assert rep["near_ties"] <= 1


def test_occupancy_variant_without_grid_table(gpu, oracle):
    """d = 4096 with G = 256 (c5's shape): the launcher drops the grid table and packs the lattice
    counts to fit one more CTA per SM; results as the definition."""
    W = wlm.random_weights(24, 4096, 82, "normal")
    rep = check(oracle, W, 4, 256, 8)
    assert rep["near_ties"] <= 2


@pytest.mark.parametrize("C,d", [(1217, 4096), (1301, 3072)])
def test_tensor_memory_rows(gpu, oracle, C, d):
    """Layers with over a thousand long channels (4096: c5's shape; 3072: 24 columns per group) at
    G = 256 keep every channel's residual row in tensor memory (4-warp groups, four CTAs per SM;
    the last CTA's second group has no channel and writes nothing).  Sampled channels against the
    definition, with a constant row (every element beside a lattice point: the queue of such
    elements overflows and the exact per-element rule runs), subnormal weights whose smallest grid
    scales round to 0 (direct evaluation), a NaN and an infinity among them."""
    W = wlm.random_weights(C, d, 83 + d, "normal")
    W[0] = np.float32(1.0)
    W[1] *= np.float32(2.0 ** -140)
    W[2, 17] = np.nan
    W[3, d - 96] = np.inf
    gpu_out = run_gpu(W, 4, 256, 4)
    sample = np.array([0, 1, 2, 3, 4, 5, 600, C - 2, C - 1])
    orc = oracle.quantize_layer(W[sample], 4, 256, 4)
    got = dict(codes=gpu_out["codes"][:, sample], scales=gpu_out["scales"][sample],
               resid_sq=gpu_out["resid_sq"][sample], residuals=gpu_out["residuals"][:, sample])
    rep = compare_quantize(W[sample], got, orc, 4, 256, 4, oracle=oracle)
    assert rep["near_ties"] <= 1
    assert np.all(np.isnan(gpu_out["scales"][2])) and np.all(gpu_out["codes"][:, 2] == 0)
    assert np.all(np.isnan(gpu_out["scales"][3])) and np.all(gpu_out["codes"][:, 3] == 0)


@pytest.mark.parametrize("bits", [2, 3, 4, 5, 6, 7, 8])
def test_bit_widths(gpu, oracle, bits):
    W = wlm.random_weights(16, 200, 50 + bits, "laplace")
    check(oracle, W, bits, 32, 3)


@pytest.mark.parametrize("G", [1, 2, 7, 31, 64, 128, 255, 256, 1024])
def test_grid_sizes(gpu, oracle, G):
    W = wlm.random_weights(8, 130, 70 + G, "t")
    check(oracle, W, 4, G, 3)


@pytest.mark.parametrize("k_max", [1, 2, 8, 16])
def test_point_counts(gpu, oracle, k_max):
    W = wlm.random_weights(6, 97, 90 + k_max, "normal")
    check(oracle, W, 3, 48, k_max)


def test_custom_grid(gpu, oracle):
    W = wlm.random_weights(12, 300, 5, "normal")
    gf = np.sort(np.random.default_rng(1).uniform(0.05, 1.0, 40)).astype(np.float32)
    gf = np.unique(gf)
    check(oracle, W, 4, gf.size, 4, grid_frac=gf)


def test_config1_full(gpu, oracle):
    """The single conv-shaped layer workload (64 x 576, b = 4, G = 64, k_max = 4) in full."""
    wl = wlm.WORKLOADS["c1"]
    W = wlm.make_weights(wl, 0)
    rep = check(oracle, W, 4, wl.G, wl.k_max)
    assert rep["checked_steps"] >= 64 * 4 - 8


def test_edge_values(gpu, oracle):
    """Zero rows, NaN/Inf rows, tiny and huge magnitudes, denormals, exact representations."""
    d = 40
    W = wlm.random_weights(10, d, 3, "normal")
    W[0] = 0.0
    W[1, 5] = np.nan
    W[2, 7] = np.inf
    W[3] *= np.float32(2.0 ** -120)   # subnormal range
    W[4] *= np.float32(2.0 ** 60)
    W[5] = (np.arange(d) % 15 - 7) * np.float32(0.25)       # exactly representable
    W[6, :] = 0.0
    W[6, 3] = -1e-40                                          # single denormal
    W[7] = np.float32(1.0)                                    # constant row
    W[8, ::2] = 0.0
    gpu_out = run_gpu(W, 4, 64, 4)
    orc = oracle.quantize_layer(W, 4, 64, 4)
    compare_quantize(W, gpu_out, orc, 4, 64, 4, oracle=oracle)
    assert np.all(np.isnan(gpu_out["scales"][1])) and np.all(gpu_out["codes"][:, 1] == 0)
    assert np.all(gpu_out["scales"][0] == 0)


def test_scale_equivariance_on_gpu(gpu):
    W = wlm.random_weights(16, 150, 3, "t")
    a = run_gpu(W, 4, 128, 6)
    b = run_gpu(np.ldexp(W, 17).astype(np.float32), 4, 128, 6)
    assert np.array_equal(a["codes"], b["codes"])
    assert np.array_equal(np.ldexp(a["scales"], 17).astype(np.float32), b["scales"])


def test_nullable_outputs_and_stream(gpu):
    W = torch.from_numpy(wlm.random_weights(5, 64, 8, "normal")).to(gpu)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        c1, s1, _, _ = binding.mpq_quantize_layer(W, 4, 32, 3, want_resid_sq=False)
    s.synchronize()
    c2, s2, _, _ = binding.mpq_quantize_layer(W, 4, 32, 3)
    torch.cuda.synchronize()
    assert torch.equal(c1, c2) and torch.equal(s1, s2)
