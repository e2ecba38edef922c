"""Parity of mpq_output_error (Eq. 11) with the oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm
from _parity import compare_err

pytestmark = pytest.mark.gpu


def gpu_err(X, W, codes, scales, k_max, groups=1, dev="cuda:0"):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    err = binding.mpq_output_error(t(X), t(W), t(codes), t(scales), k_max, groups=groups)
    torch.cuda.synchronize()
    return err.cpu().numpy()


@pytest.mark.parametrize("C,d,N,K", [(1, 1, 1, 1), (3, 5, 7, 2), (5, 33, 70, 4), (7, 64, 64, 3),
                                     (11, 147, 129, 4), (4, 1000, 65, 2), (64, 576, 512, 4),
                                     (2, 17, 300, 16),
                                     # d % 16 == 0 (CTA-pair kernel): several pair tiles with a
                                     # part-filled last pair, an empty odd CTA, ragged row tiles
                                     # split over a cluster, k_max + 1 from 2 to 17
                                     (130, 256, 600, 4), (30, 128, 1000, 1), (9, 32, 300, 16),
                                     (50, 512, 1100, 6), (3, 48, 20, 8),
                                     # k_max + 1 = 8 and 16: no channel pairing separates the
                                     # stores' bank halves there (layout unchanged, results too)
                                     (40, 96, 300, 7), (17, 64, 260, 15),
                                     (3, 8192, 300, 4)])          # the longest rows taken
def test_shared_input(gpu, oracle, C, d, N, K):
    W = wlm.random_weights(C, d, C + d + N, "normal")
    q = oracle.quantize_layer(W, 4, 32, K)
    X = wlm.random_calibration(N, d, 7 + d)
    e_or = oracle.output_error(X, 1, W, q["codes"], q["scales"], K)
    e_gpu = gpu_err(X, W, q["codes"], q["scales"], K)
    compare_err(e_gpu, e_or)


@pytest.mark.parametrize("C,d,N,K", [(1, 9, 1, 1), (6, 9, 100, 8), (40, 9, 1024, 8), (3, 25, 77, 4),
                                     (5, 300, 33, 16)])
def test_per_channel_input(gpu, oracle, C, d, N, K):
    W = wlm.random_weights(C, d, 3 * C + d, "laplace")
    q = oracle.quantize_layer(W, 4, 64, K)
    X = wlm.random_calibration(N, d, 11, groups=C)
    e_or = oracle.output_error(X, C, W, q["codes"], q["scales"], K)
    e_gpu = gpu_err(X, W, q["codes"], q["scales"], K, groups=C)
    compare_err(e_gpu, e_or)


def test_config1_layer(gpu, oracle):
    wl = wlm.WORKLOADS["c1"]
    W = wlm.make_weights(wl, 0)
    X = wlm.make_calibration(wl, 0)
    q = oracle.quantize_layer(W, 4, wl.G, wl.k_max)
    worst = compare_err(gpu_err(X, W, q["codes"], q["scales"], wl.k_max),
                        oracle.output_error(X, 1, W, q["codes"], q["scales"], wl.k_max))
    assert worst < 1e-5


def test_hot_columns_input(gpu, oracle):
    """Inputs with a few large columns (the large-linear-layer workload's calibration recipe)."""
    rng = np.random.default_rng(4)
    X = rng.standard_normal((256, 512)).astype(np.float32)
    X[:, rng.choice(512, 8, replace=False)] *= 10
    W = (rng.standard_normal((24, 512)) * 0.02).astype(np.float32)
    q = oracle.quantize_layer(W, 4, 256, 8)
    compare_err(gpu_err(X, W, q["codes"], q["scales"], 8),
                oracle.output_error(X, 1, W, q["codes"], q["scales"], 8))


def test_nonfinite_weight_propagates(gpu, oracle):
    W = wlm.random_weights(3, 20, 1, "normal")
    W[1, 2] = np.nan
    q = oracle.quantize_layer(W, 4, 16, 2)
    X = wlm.random_calibration(10, 20, 2)
    e = gpu_err(X, W, q["codes"], q["scales"], 2)
    assert np.all(np.isnan(e[1])) and np.all(np.isfinite(e[[0, 2]]))


@pytest.mark.parametrize("x_exp,w_exp", [(40, -60), (-50, 30), (0, -40)])
def test_operand_scaling_extremes(gpu, oracle, x_exp, w_exp):
    """fp16 operands are scaled per residual vector and per layer of X: inputs scaled by powers of
    two far from 1 (the oracle's double result scales exactly), residuals that reach 0 after one
    point, and calibration rows many binades below the others."""
    C, d, N, K = 40, 256, 300, 6
    W = wlm.random_weights(C, d, 3, "normal")
    W[5] = np.ldexp(np.round(W[5] * 64), -8).astype(np.float32)    # few distinct values
    W[6] = 0.0
    X = wlm.random_calibration(N, d, 4)
    X[::7] *= np.float32(2.0 ** -30)
    W = np.ldexp(W, w_exp).astype(np.float32)
    X = np.ldexp(X, x_exp).astype(np.float32)
    q = oracle.quantize_layer(W, 4, 32, K)
    compare_err(gpu_err(X, W, q["codes"], q["scales"], K),
                oracle.output_error(X, 1, W, q["codes"], q["scales"], K))


def test_nonfinite_on_the_pair_path(gpu, oracle):
    """Rows a multiple of 16 (scaled fp16 operands): the range pass skips NaN in its maxima, and
    the NaN still propagates -- a NaN weight into its channel's errors only, a NaN calibration
    input into every error."""
    W = wlm.random_weights(40, 64, 5, "normal")
    W[7, 3] = np.nan
    q = oracle.quantize_layer(W, 4, 16, 3)
    X = wlm.random_calibration(300, 64, 6)
    e = gpu_err(X, W, q["codes"], q["scales"], 3)
    assert np.all(np.isnan(e[7])) and np.all(np.isfinite(np.delete(e, 7, axis=0)))
    compare_err(e, oracle.output_error(X, 1, W, q["codes"], q["scales"], 3))
    X[100, 10] = np.nan
    assert np.all(np.isnan(gpu_err(X, W, q["codes"], q["scales"], 3)))


@pytest.mark.parametrize("C,d,N,K,bits", [(130, 256, 600, 4, 4), (64, 576, 1024, 8, 4),
                                          (9, 32, 300, 16, 3), (3, 147, 100, 4, 4)])
def test_ranges_from_the_greedy_search(gpu, oracle, C, d, N, K, bits):
    """mpq_quantize_layer's rmax output is max |r| of every residual vector (w, then each step's
    residual, exactly as the oracle's recursion gives them), and mpq_output_error with it gives
    bit for bit the errors it gives measuring the ranges itself (also for rows the tensor-core
    path cannot take, which ignore it), within 1e-5 of the oracle."""
    W = wlm.random_weights(C, d, 3 * C + d, "normal")
    W[1, 3] = np.nan                                   # a non-finite channel: NaN ranges
    X = wlm.random_calibration(N, d, 11 + d)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    rmax = torch.empty((C, K + 1), dtype=torch.float32, device=gpu)
    codes, scales, _, _ = binding.mpq_quantize_layer(t(W), bits, 64, K, rmax=rmax)
    e1 = binding.mpq_output_error(t(X), t(W), codes, scales, K, rmax=rmax)
    e0 = binding.mpq_output_error(t(X), t(W), codes, scales, K)
    torch.cuda.synchronize()
    o = oracle.quantize_layer(W, bits, 64, K)
    want = np.concatenate([np.abs(W).max(axis=1, keepdims=True),
                           np.abs(o["residuals"]).max(axis=2).T], axis=1)
    want[1, :] = np.nan
    np.testing.assert_array_equal(rmax.cpu().numpy(), want.astype(np.float32))
    assert torch.equal(torch.nan_to_num(e1, nan=-1.0), torch.nan_to_num(e0, nan=-1.0))
    keep = np.arange(C) != 1
    e_or = oracle.output_error(X, 1, W[keep], o["codes"][:, keep], o["scales"][keep], K)
    compare_err(e1.cpu().numpy()[keep], e_or)
