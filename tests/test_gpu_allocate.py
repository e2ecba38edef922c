"""Parity of mpq_allocate_points (Algorithm 2) and mpq_reconstruct (Eq. 4) with the oracle."""
import json
import os

import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def gpu_alloc(err, k_max, mode, val, dev="cuda:0"):
    e = torch.from_numpy(np.ascontiguousarray(err, np.float32)).to(dev)
    n, used = binding.mpq_allocate_points(e, k_max, mode, val)
    torch.cuda.synchronize()
    return n.cpu().numpy(), int(used.cpu().item())


def tables():
    rng = np.random.default_rng(0)
    out = []
    for C, K in ((1, 1), (1, 2), (3, 3), (17, 4), (100, 6), (1000, 8), (5000, 4), (11008, 8),
                 (300, 16)):
        e = np.sort(rng.random((C, K + 1)), 1)[:, ::-1] * rng.lognormal(0, 2, (C, 1))
        out.append(("smooth", e.astype(np.float32), K))
        ti = rng.integers(0, 6, size=(C, K + 1)).astype(np.float32)   # ties, zero/negative gains
        out.append(("ties", ti, K))
        ti2 = np.cumsum(rng.integers(0, 3, size=(C, K + 1))[:, ::-1], 1)[:, ::-1].astype(np.float32)
        out.append(("monotone_ties", ti2, K))
    return out


@pytest.mark.parametrize("case", range(27))
@pytest.mark.parametrize("beta", [0.5, 1.0, 1.25, 1.3, 1.5, 2.0, 3.7, 100.0])
def test_budget_matches_sequential_loop(gpu, oracle, case, beta):
    name, err, K = tables()[case]
    n_or, used_or = oracle.allocate_budget(err, K, beta)
    n_gpu, used_gpu = gpu_alloc(err, K, binding.MPQ_ALLOC_BUDGET, beta)
    assert np.array_equal(n_gpu, n_or), name
    assert used_gpu == used_or


@pytest.mark.parametrize("case", range(27))
def test_threshold_matches_algorithm2(gpu, oracle, case):
    name, err, K = tables()[case]
    for eps in (0.0, float(np.median(err)), 1.0, 3.0, float("inf")):
        n_or, used_or = oracle.allocate_threshold(err, K, eps)
        n_gpu, used_gpu = gpu_alloc(err, K, binding.MPQ_ALLOC_THRESHOLD, eps)
        assert np.array_equal(n_gpu, n_or), (name, eps)
        assert used_gpu == used_or


def test_allocation_hand_example_on_gpu(gpu):
    ex = json.load(open(os.path.join(GOLDEN, "allocation_hand_example.json")))
    err = np.array(ex["err"], np.float32)
    for case in ex["budget_cases"]:
        n, used = gpu_alloc(err, ex["k_max"], binding.MPQ_ALLOC_BUDGET, case["beta"])
        assert n.tolist() == case["npoints"] and used == case["used"]
    for case in ex["threshold_cases"]:
        n, used = gpu_alloc(err, ex["k_max"], binding.MPQ_ALLOC_THRESHOLD, case["eps"])
        assert n.tolist() == case["npoints"] and used == case["used"]


def test_nan_gains(gpu, oracle):
    err = np.array([[5, 4, np.nan, 1], [5, 3, 2, 1], [np.nan] * 4], np.float32)
    for beta in (1.0, 2.0, 3.0):
        n_or, u_or = oracle.allocate_budget(err, 3, beta)
        n_gpu, u_gpu = gpu_alloc(err, 3, binding.MPQ_ALLOC_BUDGET, beta)
        assert np.array_equal(n_gpu, n_or) and u_gpu == u_or


@pytest.mark.parametrize("C,d,K", [(1, 1, 1), (3, 7, 4), (64, 576, 4), (5, 1001, 8), (2, 12, 16)])
def test_reconstruct_bit_exact(gpu, oracle, C, d, K):
    W = wlm.random_weights(C, d, C * d, "normal")
    q = oracle.quantize_layer(W, 4, 64, K)
    rng = np.random.default_rng(C)
    npts = rng.integers(-1, K + 2, size=C).astype(np.int32)   # includes out-of-range (clamped)
    ref = oracle.reconstruct(q["codes"], q["scales"], npts)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    out = binding.mpq_reconstruct(t(q["codes"]), t(q["scales"]), t(npts)).cpu().numpy()
    assert np.array_equal(out, ref)


def test_reconstruct_equals_weight_minus_residual(gpu, oracle):
    """Eq. 4 and Eq. 7 together: with n = k_max points, w - w~ equals the last residual up to the
    fp32 roundings of the two recursions (<= k_max ulps of max|w|)."""
    W = wlm.random_weights(8, 256, 77, "normal")
    q = oracle.quantize_layer(W, 4, 64, 4)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    What = binding.mpq_reconstruct(t(q["codes"]), t(q["scales"]),
                                   t(np.full(8, 4, np.int32))).cpu().numpy()
    ulp = np.spacing(np.abs(W).max(1, keepdims=True).astype(np.float32))
    assert np.all(np.abs(W.astype(np.float64) - What - q["residuals"][3]) <= 4 * ulp)


@pytest.mark.parametrize("K", [4, 8])
@pytest.mark.parametrize("mode", [0, 1])
def test_batched_allocation_matches_per_layer(gpu, oracle, K, mode):
    """mpq_allocate_points_batched: every layer's point counts and total equal the oracle's
    Algorithm 2 for that layer (budget or threshold, its own beta / eps), for layers of very
    different sizes in one launch (an empty one included), tie-heavy tables among them."""
    rng = np.random.default_rng(K + 10 * mode)
    sizes = [64, 1, 0, 512, 1000, 7, 2048, 300, 11008, 33]
    errs, vals = [], []
    for i, C in enumerate(sizes):
        if i % 3 == 1:
            e = rng.integers(0, 6, size=(C, K + 1)).astype(np.float32)
        else:
            e = (np.sort(rng.random((C, K + 1)), 1)[:, ::-1] *
                 rng.lognormal(0, 2, (C, 1))).astype(np.float32)
        errs.append(np.ascontiguousarray(e))
        vals.append([1.0, 1.25, 1.5, 2.0, 3.7][i % 5] if mode == 0 else
                    float(np.median(e)) if C else 0.5)
    t = [torch.from_numpy(e).to(gpu) for e in errs]
    n_gpu, used_gpu = binding.mpq_allocate_points_batched(t, K, mode, vals)
    torch.cuda.synchronize()
    for e, v, n, u in zip(errs, vals, n_gpu, used_gpu):
        if mode == 0:
            n_or, used_or = oracle.allocate_budget(e, K, v)
        else:
            n_or, used_or = oracle.allocate_threshold(e, K, v)
        assert np.array_equal(n.cpu().numpy(), n_or)
        assert int(u.item()) == used_or


@pytest.mark.parametrize("C,K", [(2048, 4), (6144, 2), (1536, 5)])
def test_budget_keys_at_the_default_shared_memory_limit(gpu, oracle, C, K):
    """C (k_max - 1) keys of exactly 48 KB (the kernel's own shared memory comes on top): the
    launch raises its shared-memory limit instead of failing."""
    rng = np.random.default_rng(C + K)
    err = (np.sort(rng.random((C, K + 1)), 1)[:, ::-1] * rng.lognormal(0, 1, (C, 1))).astype(np.float32)
    n_or, used_or = oracle.allocate_budget(err, K, 1.5)
    n_gpu, used_gpu = gpu_alloc(err, K, binding.MPQ_ALLOC_BUDGET, 1.5)
    assert np.array_equal(n_gpu, n_or) and used_gpu == used_or
