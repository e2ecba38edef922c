"""Integer inference with multipoint weights (Eq. 13, Sec. 3.4) through the C ABI: packing and the
tensor-core / integer kernels bit-exact against the oracle's exact integer arithmetic."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def points(C, k_max, seed, mix=None):
    rng = np.random.default_rng(seed)
    if mix is None:
        return rng.integers(0, k_max + 1, C).astype(np.int32)
    return rng.choice(np.array(mix, np.int32), C).astype(np.int32)


def run(oracle, codes, scales, npts, X, bits, p):
    k_max, C, d = codes.shape
    lay = binding.mpq_pack_layout(npts, d, k_max, bits, p)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    packed = binding.mpq_pack_points(t(codes), t(scales), npts, lay)
    Y = binding.mpq_multipoint_linear(t(X), lay, packed)
    torch.cuda.synchronize()
    return Y.cpu().numpy(), lay


@pytest.mark.parametrize("C,d,T,k_max,bits,p,mix", [
    (200, 256, 300, 4, 4, 12, None),               # every n_k in 0..4: groups R = 1, 2, 4
    (333, 512, 1, 8, 4, 16, [1, 1, 1, 2, 3, 5]),    # one input row, R up to 8
    (64, 64, 513, 16, 4, 20, [16, 9, 1]),           # R = 16, three 256-input tiles (ragged)
    (1000, 1152, 100, 4, 4, 0, [1, 2]),             # p = 0
    (130, 96, 700, 6, 3, 24, None),                 # 3-bit codes, d not a multiple of 64
    (20, 8192, 300, 2, 4, 16, None),                # the longest rows (8192 x 7 x 128 < 2^24)
])
def test_tensor_path(gpu, oracle, C, d, T, k_max, bits, p, mix):
    W = wlm.random_weights(C, d, C + d, "laplace")
    q = oracle.quantize_layer(W, bits, 32, k_max, threads=8)
    npts = points(C, k_max, C + T, mix)
    X = np.random.default_rng(T).integers(-128, 128, (T, d)).astype(np.int8)
    Y, lay = run(oracle, q["codes"], q["scales"], npts, X, bits, p)
    assert np.array_equal(Y, oracle.multipoint_linear(X, q["codes"], q["scales"], npts, p,
                                                      threads=8))


@pytest.mark.parametrize("C,d,T,k_max,bits,p", [
    (11, 147, 129, 4, 4, 12),     # rows not 16-byte multiples: integer kernel
    (9, 2048, 33, 2, 8, 10),      # 8-bit codes: 2048 * 127 * 128 >= 2^24, integer kernel
])
def test_integer_path(gpu, oracle, C, d, T, k_max, bits, p):
    W = wlm.random_weights(C, d, 5 + d, "normal")
    q = oracle.quantize_layer(W, bits, 16, k_max)
    npts = points(C, k_max, 9)
    X = np.random.default_rng(3).integers(-128, 128, (T, d)).astype(np.int8)
    Y, _ = run(oracle, q["codes"], q["scales"], npts, X, bits, p)
    assert np.array_equal(Y, oracle.multipoint_linear(X, q["codes"], q["scales"], npts, p))


def test_saturation_and_extremes(gpu, oracle):
    """Codes and inputs at their extremes (|q| = Qmax, x = -128) and large coefficients."""
    k_max, C, d, T = 3, 40, 128, 260
    codes = np.where(np.random.default_rng(1).random((k_max, C, d)) < 0.5, 7, -7).astype(np.int8)
    scales = np.full((C, k_max), 3000.0, np.float32)
    npts = points(C, k_max, 2)
    X = np.full((T, d), -128, np.int8)
    X[::3] = 127
    for p in (0, 16):
        Y, _ = run(oracle, codes, scales, npts, X, 4, p)
        assert np.array_equal(Y, oracle.multipoint_linear(X, codes, scales, npts, p))


def test_coefficient_overflow_is_reported(gpu):
    codes = torch.zeros((1, 2, 32), dtype=torch.int8, device=DEV)
    scales = torch.tensor([[1000.0], [0.5]], device=DEV)
    lay = binding.mpq_pack_layout([1, 1], 32, 1, 4, 22)
    with pytest.raises(binding.MPQError) as e:
        binding.mpq_pack_points(codes, scales, [1, 1], lay)
    assert e.value.status == 3


def test_full_size_sampled(gpu, oracle):
    """c5's up_proj (11008 x 4096) quantized and allocated on the device, 2048 int8 inputs through
    the tensor-core kernel, checked on sampled channels against the oracle."""
    wl = wlm.WORKLOADS["c5"]
    W = torch.from_numpy(wlm.make_weights(wl, 1)).to(DEV)
    codes, scales, _, _ = binding.mpq_quantize_layer(W, 4, wl.G, wl.k_max)
    Xc = torch.from_numpy(wlm.make_calibration(wl, 1)).to(DEV)
    err = binding.mpq_output_error(Xc, W, codes, scales, wl.k_max)
    npts, _ = binding.mpq_allocate_points(err, wl.k_max, binding.MPQ_ALLOC_BUDGET, wl.beta)
    n_host = npts.cpu().numpy()
    X = np.random.default_rng(7).integers(-128, 128, (2048, 4096)).astype(np.int8)
    lay = binding.mpq_pack_layout(n_host, 4096, wl.k_max, 4, 16)
    packed = binding.mpq_pack_points(codes, scales, n_host, lay)
    Y = binding.mpq_multipoint_linear(torch.from_numpy(X).to(DEV), lay, packed).cpu().numpy()
    c_np, s_np = codes.cpu().numpy(), scales.cpu().numpy()
    for c0 in (0, 5000, 11008 - 16):
        ref = oracle.multipoint_linear(X, c_np, s_np, n_host, 16, channels=(c0, c0 + 16), threads=8)
        assert np.array_equal(Y[c0:c0 + 16], ref[c0:c0 + 16])
