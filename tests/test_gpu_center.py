"""Asymmetric sets (Eq. 1 with B != 0) through the C ABI: centres and centred weights bit-exact
against the oracle, the whole path on centred weights (greedy points, Eq. 11, Algorithm 2, Eq. 4
from the centre), and integer inference (Eq. 13) with the centre's A_B sum(x) term, bit-exact."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, pipeline, workloads as wlm
from _parity import compare_err, compare_quantize

pytestmark = pytest.mark.gpu

MODES = (binding.MPQ_CENTER_PER_CHANNEL, binding.MPQ_CENTER_PER_LAYER)


def t(a, dev="cuda:0"):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def offset_weights(C, d, seed, dist="laplace"):
    """Weights with a per-channel offset, so that the centres are far from 0."""
    W = wlm.random_weights(C, d, seed, dist)
    off = np.random.default_rng(seed + 1).uniform(-0.2, 0.3, (C, 1)).astype(np.float32)
    return (W + off).astype(np.float32)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("C,d", [(1, 1), (7, 33), (130, 576), (5, 8192), (3000, 9)])
def test_center_parity(gpu, oracle, mode, C, d):
    W = offset_weights(C, d, C + d)
    B, Wc = binding.mpq_center_weights(t(W), mode)
    torch.cuda.synchronize()
    oB, oWc = oracle.center(W, mode)
    assert np.array_equal(B.cpu().numpy(), oB)
    assert np.array_equal(Wc.cpu().numpy(), oWc)


def test_center_extremes(gpu, oracle):
    """Large and tiny magnitudes, a constant channel, an all-zero channel, one-sided ranges."""
    W = np.zeros((6, 40), np.float32)
    W[0] = np.linspace(-3e30, 1e30, 40)
    W[1] = np.linspace(1e-30, 5e-30, 40)
    W[2] = 0.7
    W[4] = -np.geomspace(1e-3, 10.0, 40)
    W[5] = np.random.default_rng(3).standard_normal(40) * 1e4
    for mode in MODES:
        B, Wc = binding.mpq_center_weights(t(W), mode)
        oB, oWc = oracle.center(W, mode)
        assert np.array_equal(B.cpu().numpy(), oB) and np.array_equal(Wc.cpu().numpy(), oWc)


def test_center_nonfinite(gpu, oracle):
    W = offset_weights(4, 50, 9)
    W[2, 7] = np.inf
    B, Wc = binding.mpq_center_weights(t(W), binding.MPQ_CENTER_PER_CHANNEL)
    B, Wc = B.cpu().numpy(), Wc.cpu().numpy()
    oB, oWc = oracle.center(W, binding.MPQ_CENTER_PER_CHANNEL)
    assert np.isnan(B[2]) and np.all(np.isnan(Wc[2]))
    assert np.array_equal(B, oB, equal_nan=True) and np.array_equal(Wc, oWc, equal_nan=True)
    Bl, _ = binding.mpq_center_weights(t(W), binding.MPQ_CENTER_PER_LAYER)
    assert np.all(np.isnan(Bl.cpu().numpy()))


@pytest.mark.parametrize("mode", MODES)
def test_asymmetric_path_end_to_end(gpu, oracle, mode):
    """One conv-shaped layer (64 x 576, N = 512) through LayerPlan with centring: greedy points on
    the centred weights, their output error, the allocation and the reconstruction from B."""
    W = offset_weights(64, 576, 11)
    X = wlm.random_calibration(512, 576, 12)
    spec = pipeline.LayerSpec(C=64, d=576, N=512, bits=4, G=64, k_max=4, budget_or_eps=2.0,
                              center=mode)
    plan = pipeline.LayerPlan(spec, gpu)
    plan.run_device(t(W), t(X))
    torch.cuda.synchronize()
    oB, oWc = oracle.center(W, mode)
    assert np.array_equal(plan.center.cpu().numpy(), oB)
    orc = oracle.quantize_layer(oWc, 4, 64, 4)
    gq = dict(codes=plan.codes.cpu().numpy(), scales=plan.scales.cpu().numpy(),
              resid_sq=plan.resid_sq.cpu().numpy())
    rep = compare_quantize(oWc, gq, orc, 4, 64, 4, oracle=oracle)
    err_gpu = plan.err.cpu().numpy()
    if rep["near_ties"] == 0:
        compare_err(err_gpu, oracle.output_error(X, 1, oWc, orc["codes"], orc["scales"], 4))
        n_or, _ = oracle.allocate_budget(err_gpu, 4, 2.0)
        assert np.array_equal(plan.npoints.cpu().numpy(), n_or)
        W_hat = oracle.reconstruct(orc["codes"], orc["scales"], n_or, center=oB)
        assert np.array_equal(plan.W_hat.cpu().numpy(), W_hat)


def run_linear(oracle, W, mode, X, bits, p, k_max, seed):
    C, d = W.shape
    B, Wc = binding.mpq_center_weights(t(W), mode)
    codes, scales, _, _ = binding.mpq_quantize_layer(Wc, bits, 32, k_max)
    npts = np.random.default_rng(seed).integers(0, k_max + 1, C).astype(np.int32)
    lay = binding.mpq_pack_layout(npts, d, k_max, bits, p, centered=True)
    packed = binding.mpq_pack_points(codes, scales, npts, lay, center=B)
    Y = binding.mpq_multipoint_linear(t(X), lay, packed).cpu().numpy()
    ref = oracle.multipoint_linear(X, codes.cpu().numpy(), scales.cpu().numpy(), npts, p,
                                   threads=8, center=B.cpu().numpy())
    return Y, ref


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("C,d,T,k_max,bits,p", [
    (200, 256, 300, 4, 4, 12),      # tensor-core kernel, groups R = 1, 2, 4, ragged inputs
    (64, 64, 513, 8, 4, 20),        # three input tiles, R up to 8
    (130, 96, 700, 6, 3, 0),        # p = 0, d not a multiple of 64
    (11, 147, 129, 4, 4, 12),       # rows not 16-byte multiples: integer kernel
    (9, 2048, 33, 2, 8, 10),        # beyond the fp32 exactness bound: integer kernel
])
def test_multipoint_linear_centered(gpu, oracle, mode, C, d, T, k_max, bits, p):
    W = offset_weights(C, d, 5 * C + d, "normal")
    X = np.random.default_rng(T).integers(-128, 128, (T, d)).astype(np.int8)
    Y, ref = run_linear(oracle, W, mode, X, bits, p, k_max, C + T)
    assert np.array_equal(Y, ref)


def test_multipoint_linear_centered_extremes(gpu, oracle):
    """Inputs at -128, large centres (A_B near 2^31 at p = 0) and saturation of the result."""
    W = offset_weights(40, 128, 21) * 1e6
    X = np.full((260, 128), -128, np.int8)
    X[::3] = 127
    for p in (0, 4):
        Y, ref = run_linear(oracle, W, binding.MPQ_CENTER_PER_CHANNEL, X, 4, p, 3, 22)
        assert np.array_equal(Y, ref)


def test_center_coefficient_overflow_is_reported(gpu):
    W = torch.full((2, 32), 3000.0, device="cuda:0")
    W[:, 0] = 3001.0
    B, Wc = binding.mpq_center_weights(W)
    codes, scales, _, _ = binding.mpq_quantize_layer(Wc, 4, 8, 1)
    lay = binding.mpq_pack_layout([1, 1], 32, 1, 4, 20, centered=True)   # 2^20 x 3000 > 2^31
    with pytest.raises(binding.MPQError) as e:
        binding.mpq_pack_points(codes, scales, [1, 1], lay, center=B)
    assert e.value.status == 3


def test_full_size_sampled(gpu, oracle):
    """c5's up_proj (11008 x 4096) centred per channel, quantized and allocated on the device,
    2048 int8 inputs through the tensor-core kernel with the centre term, checked on sampled
    channels against the oracle."""
    wl = wlm.WORKLOADS["c5"]
    W = torch.from_numpy(wlm.make_weights(wl, 1)).to(gpu)
    B, Wc = binding.mpq_center_weights(W, binding.MPQ_CENTER_PER_CHANNEL)
    oB, _ = oracle.center(W.cpu().numpy(), binding.MPQ_CENTER_PER_CHANNEL)
    assert np.array_equal(B.cpu().numpy(), oB)
    codes, scales, _, _ = binding.mpq_quantize_layer(Wc, 4, wl.G, wl.k_max)
    Xc = torch.from_numpy(wlm.make_calibration(wl, 1)).to(gpu)
    err = binding.mpq_output_error(Xc, Wc, codes, scales, wl.k_max)
    npts, _ = binding.mpq_allocate_points(err, wl.k_max, binding.MPQ_ALLOC_BUDGET, wl.beta)
    n_host = npts.cpu().numpy()
    X = np.random.default_rng(8).integers(-128, 128, (2048, 4096)).astype(np.int8)
    lay = binding.mpq_pack_layout(n_host, 4096, wl.k_max, 4, 16, centered=True)
    packed = binding.mpq_pack_points(codes, scales, n_host, lay, center=B)
    Y = binding.mpq_multipoint_linear(t(X), lay, packed).cpu().numpy()
    c_np, s_np = codes.cpu().numpy(), scales.cpu().numpy()
    for c0 in (0, 7000, 11008 - 16):
        ref = oracle.multipoint_linear(X, c_np, s_np, n_host, 16, channels=(c0, c0 + 16), threads=8,
                                       center=oB)
        assert np.array_equal(Y[c0:c0 + 16], ref[c0:c0 + 16])
