"""Pins of the CPU oracle to facts fixed by the paper and by mathematics (no GPU needed).

Each test checks the oracle against something other than itself: a hand-worked example, exhaustive
enumeration, a closed form, an invariance of the method, or a library routine used as a step.
"""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from paper_2002_09049_gb300 import workloads as wlm

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _grid(m, qmax, G, grid_frac=None):
    """The candidate-scale grid as stated in the method description (fp32)."""
    smax = np.float32(m) / np.float32(qmax)
    f = (np.arange(1, G + 1, dtype=np.float32) / np.float32(G)) if grid_frac is None else \
        np.asarray(grid_frac, np.float32)
    return (f * smax).astype(np.float32)


# --- Algorithm 1 / Eq. 7-9 --------------------------------------------------------------------

def test_hand_worked_example(oracle):
    """Sec. 3.2 Eq. 7-9: matches a two-step example worked by hand."""
    ex = json.load(open(os.path.join(GOLDEN, "greedy_hand_example.json")))
    W = np.array([ex["w"]], np.float32)
    out = oracle.quantize_layer(W, ex["bits"], ex["G"], ex["k_max"])
    r = W[0].copy()
    for i, st in enumerate(ex["steps"]):
        E, s = oracle.candidate_errors(r, ex["bits"], ex["G"])
        np.testing.assert_allclose(s, st["scales"], rtol=1e-6)
        np.testing.assert_allclose(E, st["E"], rtol=1e-6)
        assert out["gstar"][0, i] == st["gstar"]
        assert out["codes"][i, 0].tolist() == st["codes"]
        np.testing.assert_allclose(out["residuals"][i, 0], st["residual_after"], atol=1e-7)
        r = out["residuals"][i, 0]


@pytest.mark.parametrize("bits,d", [(2, 1), (2, 2), (2, 3), (2, 4), (3, 2), (3, 3)])
@pytest.mark.parametrize("seed", range(6))
def test_brute_force_step_is_grid_optimal(oracle, bits, d, seed):
    """Eq. 8-9: for every grid scale the rounded codes are the best code vector (exhaustive over
    all (2Qmax+1)^d vectors), and the chosen scale attains the exhaustive minimum over
    (scale, code).  The one allowed slack: the codes come from an fp32 quotient r/s, so an element
    whose exact r/s lies within half an fp32 ulp of a half-integer may take the other neighbour,
    costing at most 2 s^2 (Qmax+1) 2^-24 of error per element."""
    qmax = 2 ** (bits - 1) - 1
    G = 16
    W = wlm.random_weights(1, d, 100 + seed, "normal")
    out = oracle.quantize_layer(W, bits, G, 3)
    r = W[0].copy()
    levels = range(-qmax, qmax + 1)
    for i in range(3):
        m = np.abs(r).max()
        if m == 0:
            assert out["scales"][0, i] == 0
            break
        scales = _grid(m, qmax, G)
        rd = r.astype(np.float64)
        exhaustive = []
        for s in scales:
            best = min(float(np.sum((rd - float(s) * np.array(q, np.float64)) ** 2))
                       for q in itertools.product(levels, repeat=d))
            exhaustive.append(best)
        exhaustive = np.array(exhaustive)
        slack = d * 2.0 * scales.astype(np.float64) ** 2 * (qmax + 1) * 2.0 ** -24
        E, s_or = oracle.candidate_errors(r, bits, G)
        np.testing.assert_array_equal(s_or, scales)
        assert np.all(E >= exhaustive * (1 - 1e-14))
        assert np.all(E - exhaustive <= slack + 1e-14 * exhaustive)
        g = out["gstar"][0, i]
        assert g == int(np.argmin(E))                       # first minimiser
        assert E[g] <= exhaustive.min() + slack[g] + 1e-14 * exhaustive.min()
        assert out["scales"][0, i] == scales[g]
        r = out["residuals"][i, 0]


def test_one_point_is_plain_per_channel_quantization(oracle):
    """Eq. 9 with n = 1: the first point is ordinary symmetric per-channel b-bit quantization with
    the best scale of the grid (vectorised textbook quantizer over all candidate scales at once)."""
    for bits, G, dist in ((4, 64, "normal"), (3, 32, "laplace"), (8, 16, "t")):
        qmax = 2 ** (bits - 1) - 1
        W = wlm.random_weights(24, 97, 7 + bits, dist)
        out = oracle.quantize_layer(W, bits, G, 1)
        for k in range(W.shape[0]):
            w = W[k]
            s = _grid(np.abs(w).max(), qmax, G)                        # [G]
            q = np.clip(np.rint(w[None, :] / s[:, None]), -qmax, qmax)  # [G, d]
            err = ((w[None, :].astype(np.float64) - s[:, None].astype(np.float64) * q) ** 2).sum(1)
            g = int(np.argmin(err))
            assert out["scales"][k, 0] == s[g]
            np.testing.assert_array_equal(out["codes"][0, k], q[g].astype(np.int8))


def test_residual_norm_non_increasing_and_strict(oracle):
    """Eq. 7 with the scale search of Eq. 9: ||r_{i+1}|| <= ||r_i||, strictly while r_i != 0
    (at the largest grid scale the largest element is represented, so some candidate improves)."""
    for dist in ("normal", "laplace", "t"):
        W = wlm.random_weights(32, 200, 11, dist)
        out = oracle.quantize_layer(W, 4, 64, 8)
        rs = out["resid_sq"]
        step = np.diff(rs, axis=1)
        assert np.all(step <= 0)
        assert np.all((step < 0) | (rs[:, :-1] == 0))


def test_exponential_decay_theorem1(oracle):
    """Theorem 1 (b = 2, fine grid): ||r_i||^2 decays geometrically; every step removes at least a
    fixed fraction of the residual energy for the first steps."""
    W = wlm.random_weights(8, 32, 5, "normal")
    out = oracle.quantize_layer(W, 2, 4096, 10)
    ratios = out["resid_sq"][:, 1:] / out["resid_sq"][:, :-1]
    assert np.all(ratios < 0.9)
    # log-linear: after 10 points the energy is down by orders of magnitude
    assert np.all(out["resid_sq"][:, -1] < 1e-3 * out["resid_sq"][:, 0])


def test_scale_equivariance(oracle):
    """The method is scale-equivariant: w -> 2^k w multiplies every scale by 2^k and leaves every
    code unchanged, bit for bit (all fp32 operations commute with exact power-of-two scaling)."""
    W = wlm.random_weights(16, 150, 3, "t")
    base = oracle.quantize_layer(W, 4, 128, 6)
    for k in (-20, -3, 5, 30):
        out = oracle.quantize_layer(np.ldexp(W, k).astype(np.float32), 4, 128, 6)
        np.testing.assert_array_equal(out["codes"], base["codes"])
        np.testing.assert_array_equal(out["scales"], np.ldexp(base["scales"], k).astype(np.float32))


def test_exactly_representable_channel(oracle):
    """If w = s0 * q0 with integer q0 and max|q0| = Qmax, the largest grid scale reproduces w
    exactly: the first point is exact and every later point is a null point."""
    rng = np.random.default_rng(0)
    q0 = rng.integers(-7, 8, size=(4, 33))
    q0[:, 0] = 7
    W = (q0 * 0.125).astype(np.float32)
    out = oracle.quantize_layer(W, 4, 64, 3)
    np.testing.assert_array_equal(out["codes"][0], q0.astype(np.int8))
    np.testing.assert_array_equal(out["scales"][:, 0], np.float32(0.125))
    assert np.all(out["gstar"][:, 0] == 63)
    assert np.all(out["resid_sq"][:, 1:] == 0)
    assert np.all(out["scales"][:, 1:] == 0) and np.all(out["codes"][1:] == 0)


def test_zero_and_nonfinite_channels(oracle):
    """Readings for degenerate channels: an all-zero channel gives null points; a channel with a
    NaN/Inf weight gives NaN scales and zero codes."""
    W = np.zeros((3, 5), np.float32)
    W[1] = [1, 2, 3, 4, 5]
    W[2, 3] = np.nan
    out = oracle.quantize_layer(W, 4, 8, 2)
    assert np.all(out["scales"][0] == 0) and np.all(out["codes"][:, 0] == 0)
    assert np.all(out["resid_sq"][0] == 0)
    assert np.all(np.isnan(out["scales"][2])) and np.all(out["codes"][:, 2] == 0)
    assert out["scales"][1, 0] > 0


def test_user_grid(oracle):
    """A caller-supplied grid of fractions replaces f_g = g/G: the chosen scale is one of them."""
    W = wlm.random_weights(10, 64, 21, "normal")
    gf = np.array([0.3, 0.5, 0.55, 0.7, 0.9, 1.0], np.float32)
    out = oracle.quantize_layer(W, 4, gf.size, 2, grid_frac=gf)
    for k in range(10):
        s = _grid(np.abs(W[k]).max(), 7, gf.size, gf)
        assert out["scales"][k, 0] in s


# --- Eq. 4: reconstruction ----------------------------------------------------------------------

def test_reconstruct_matches_exact_sum(oracle):
    """Eq. 4: w~(n) = sum_i s_i q_i; the fmaf chain is within n half-ulps of the exact rational
    sum, and w - w~(n) equals the residual r_{n+1} up to the same rounding."""
    W = wlm.random_weights(6, 40, 9, "normal")
    K = 4
    out = oracle.quantize_layer(W, 4, 64, K)
    for n in range(K + 1):
        npts = np.full(6, n, np.int32)
        What = oracle.reconstruct(out["codes"], out["scales"], npts)
        for k in range(6):
            for j in range(0, 40, 7):
                exact = sum(Fraction(float(out["scales"][k, i])) * int(out["codes"][i, k, j])
                            for i in range(n))
                got = Fraction(float(What[k, j]))
                ulp = float(np.spacing(np.abs(W[k]).max().astype(np.float32)))  # fp32 ulp
                assert abs(float(got - exact)) <= max(n, 1) * ulp
                if n > 0:
                    resid = Fraction(float(out["residuals"][n - 1, k, j]))
                    assert abs(float(Fraction(float(W[k, j])) - exact - resid)) <= n * ulp


# --- Eq. 11: output error -----------------------------------------------------------------------

def _quantized(oracle, C=6, d=64, K=3, seed=4):
    W = wlm.random_weights(C, d, seed, "normal")
    return W, oracle.quantize_layer(W, 4, 32, K)


def test_output_error_identity_input(oracle):
    """Eq. 11 with X = sqrt(N) I (N = d = 64): e(n) = ||r_{n+1}||^2 = resid_sq."""
    W, q = _quantized(oracle)
    X = (np.eye(64) * 8.0).astype(np.float32)
    err = oracle.output_error(X, 1, W, q["codes"], q["scales"], 3)
    np.testing.assert_allclose(err, q["resid_sq"], rtol=1e-13)


def test_output_error_single_column(oracle):
    """Eq. 11 with one nonzero input column j0 of value c: e(n) = c^2 r_{n+1,j0}^2."""
    W, q = _quantized(oracle)
    j0, c = 17, 3.0
    X = np.zeros((10, 64), np.float32)
    X[:, j0] = c
    err = oracle.output_error(X, 1, W, q["codes"], q["scales"], 3)
    R = np.concatenate([W[None], q["residuals"]], 0)   # [K+1][C][d]
    expect = (c * R[:, :, j0].astype(np.float64)) ** 2
    np.testing.assert_allclose(err, expect.T, rtol=1e-13)


def test_output_error_matches_library_matmul(oracle):
    """Eq. 11 against a double-precision library matmul of X with the residuals."""
    W, q = _quantized(oracle, C=5, d=70, K=4, seed=8)
    X = wlm.random_calibration(33, 70, 2)
    err = oracle.output_error(X, 1, W, q["codes"], q["scales"], 4)
    R = np.concatenate([W[None], q["residuals"]], 0).astype(np.float64)  # [K+1][C][d]
    Y = np.einsum("td,ncd->nct", X.astype(np.float64), R)
    np.testing.assert_allclose(err, (Y ** 2).mean(-1).T, rtol=1e-12)


def test_output_error_depthwise_blocks(oracle):
    """groups = C: channel k reads its own N x d input block (depthwise convolution)."""
    W, q = _quantized(oracle, C=4, d=9, K=3, seed=12)
    X = wlm.random_calibration(20, 9, 3, groups=4)
    err = oracle.output_error(X, 4, W, q["codes"], q["scales"], 3)
    R = np.concatenate([W[None], q["residuals"]], 0).astype(np.float64)
    for k in range(4):
        Y = X[k].astype(np.float64) @ R[:, k, :].T     # [N][K+1]
        np.testing.assert_allclose(err[k], (Y ** 2).mean(0), rtol=1e-12)


# --- Algorithm 2: point allocation --------------------------------------------------------------

def test_allocation_hand_example(oracle):
    ex = json.load(open(os.path.join(GOLDEN, "allocation_hand_example.json")))
    err = np.array(ex["err"], np.float32)
    for case in ex["budget_cases"]:
        n, used = oracle.allocate_budget(err, ex["k_max"], case["beta"])
        assert n.tolist() == case["npoints"], case["why"]
        assert used == case["used"]
    for case in ex["threshold_cases"]:
        n, used = oracle.allocate_threshold(err, ex["k_max"], case["eps"])
        assert n.tolist() == case["npoints"], case["why"]
        assert used == case["used"]


def test_allocation_budget_extremes(oracle):
    """beta = 1 gives one point everywhere; beta = k_max with positive gains gives k_max."""
    rng = np.random.default_rng(3)
    C, K = 50, 5
    err = np.sort(rng.random((C, K + 1)), axis=1)[:, ::-1].astype(np.float32) + 1
    n, used = oracle.allocate_budget(err, K, 1.0)
    assert np.all(n == 1) and used == C
    n, used = oracle.allocate_budget(err, K, float(K))
    assert np.all(n == K) and used == C * K


def test_allocation_greedy_is_optimal_for_concave_gains(oracle):
    """With diminishing returns (decreasing gains per channel) the marginal-gain loop maximises
    the total output-error reduction for its budget: exhaustive check on small tables."""
    rng = np.random.default_rng(5)
    for trial in range(20):
        C, K = 3, 4
        gains = np.sort(rng.integers(1, 50, size=(C, K - 1)), axis=1)[:, ::-1]   # decreasing
        e1 = rng.integers(200, 300, size=(C, 1))
        err = np.concatenate([e1 + 100, e1 - np.concatenate(
            [np.zeros((C, 1), int), np.cumsum(gains, 1)], 1)], 1).astype(np.float32)
        for extra in range(0, C * (K - 1) + 1):
            beta = (C + extra) / C
            n, used = oracle.allocate_budget(err, K, beta)
            best = max(sum(err[k, 1] - err[k, a[k]] for k in range(C))
                       for a in itertools.product(range(1, K + 1), repeat=C)
                       if sum(a) == C + extra)
            got = sum(err[k, 1] - err[k, n[k]] for k in range(C))
            assert used == C + extra
            assert got == best


def test_allocation_stops_at_nonpositive_gain(oracle):
    err = np.array([[5, 4, 4.5, 1], [5, 3, 3, 3]], np.float32)
    n, used = oracle.allocate_budget(err, 3, 3.0)
    # ch0 head gain 4-4.5 < 0, ch1 head gain 0: nothing is worth adding
    assert n.tolist() == [1, 1] and used == 2


# --- Table 1: overhead closed forms -------------------------------------------------------------

def test_table1_overhead_closed_forms():
    """Table 1: naive vs multipoint memory / MULs / ADDs; n = 1 reduces to naive plus the
    32-bit coefficient."""
    from paper_2002_09049_gb300 import overhead
    d, Nb = 576, 4
    naive = overhead.naive_cost(d, Nb)
    assert naive == dict(memory_bits=d * Nb, muls=d * Nb * Nb, adds=(d - 1) * Nb)
    mp = overhead.multipoint_cost(d, Nb, 3)
    assert mp == dict(memory_bits=3 * d * Nb + 96, muls=3 * (d * Nb * Nb + 1024),
                      adds=3 * (d - 1) * Nb + 64)
    one = overhead.multipoint_cost(d, Nb, 1)
    assert one["memory_bits"] - naive["memory_bits"] == 32 and one["adds"] == naive["adds"]


# ---- Eq. 12: output-error-driven clipping factor -------------------------------------------------

def test_clip_hand_example(oracle):
    """Candidates, errors and both argmins of a 2-channel example worked by hand (exact dyadics),
    including a tie between two candidates (lowest index wins)."""
    g = json.load(open(os.path.join(GOLDEN, "clip_hand_example.json")))
    W = np.array(g["W"], np.float32)
    for mode in (oracle.CLIP_PER_CHANNEL, oracle.CLIP_PER_LAYER):
        clip = oracle.clip_candidates(W, g["n_cand"], mode)
        assert np.array_equal(clip, np.tile(np.float32([0.25, 0.5, 0.75, 1.0]), (2, 1)))
    clip = oracle.clip_candidates(W, g["n_cand"], oracle.CLIP_PER_CHANNEL)
    for xs in ("X1", "X2"):
        X = np.array(g[xs], np.float32)
        e = oracle.clip_errors(X, 1, W, g["bits"], clip)
        assert np.array_equal(e, np.array(g["err_" + xs]))
        e32 = e.astype(np.float32)
        assert list(oracle.clip_select(e32, oracle.CLIP_PER_CHANNEL)) == g["best_per_channel_" + xs]
        assert list(oracle.clip_select(e32, oracle.CLIP_PER_LAYER)) == g["best_per_layer_" + xs]


def test_clip_candidates_grid_and_modes(oracle):
    rng = np.random.default_rng(31)
    W = (rng.standard_normal((5, 40)) * rng.uniform(0.1, 3.0, (5, 1))).astype(np.float32)
    per_ch = oracle.clip_candidates(W, 20, oracle.CLIP_PER_CHANNEL)
    per_l = oracle.clip_candidates(W, 20, oracle.CLIP_PER_LAYER)
    m = np.abs(W).max(axis=1)
    assert np.array_equal(per_ch[:, -1], m)                  # f = 1: K = max|w| exactly
    f = (np.arange(1, 21, dtype=np.float32) / np.float32(20)).astype(np.float32)
    assert np.array_equal(per_ch, (f[None, :] * m[:, None]).astype(np.float32))
    assert np.array_equal(per_l, np.tile((f * np.float32(m.max())).astype(np.float32), (5, 1)))


def test_clip_scale_equivariance(oracle):
    """W -> 2^k W scales every K by 2^k, every output error by 4^k, and keeps both argmins."""
    rng = np.random.default_rng(32)
    W = rng.standard_normal((6, 33)).astype(np.float32)
    X = rng.standard_normal((17, 33)).astype(np.float32)
    for mode in (oracle.CLIP_PER_CHANNEL, oracle.CLIP_PER_LAYER):
        c0 = oracle.clip_candidates(W, 20, mode)
        e0 = oracle.clip_errors(X, 1, W, 4, c0)
        for k in (-3, 5):
            W2 = np.ldexp(W, k).astype(np.float32)
            c2 = oracle.clip_candidates(W2, 20, mode)
            assert np.array_equal(c2, np.ldexp(c0, k).astype(np.float32))
            e2 = oracle.clip_errors(X, 1, W2, 4, c2)
            assert np.allclose(e2, e0 * 4.0 ** k, rtol=1e-12, atol=0)
            assert np.array_equal(oracle.clip_select(e2.astype(np.float32), mode),
                                  oracle.clip_select(e0.astype(np.float32), mode))


def test_clip_top_candidate_is_greedy_top_scale(oracle):
    """With X = sqrt(N) I, the error of K = max|w| is the weight error of the greedy search's largest
    scale (same set, same codes): the two oracle functions agree."""
    rng = np.random.default_rng(33)
    d = 24
    W = rng.standard_normal((4, d)).astype(np.float32)
    X = (np.eye(d) * np.sqrt(d)).astype(np.float32)    # N = d rows: mean_t (x_t . r)^2 = ||r||^2
    clip = oracle.clip_candidates(W, 20, oracle.CLIP_PER_CHANNEL)
    e = oracle.clip_errors(X, 1, W, 3, clip)
    for k in range(4):
        ce, sg = oracle.candidate_errors(W[k], 3, 16)
        assert sg[-1] == np.float32(clip[k, -1] / np.float32(3))   # the same scale m / Qmax
        assert np.isclose(e[k, -1], ce[-1], rtol=1e-6, atol=0)


def test_clip_select_brute_force(oracle):
    """Both argmins against brute force on tie-heavy integer tables with NaNs."""
    rng = np.random.default_rng(34)
    for _ in range(200):
        C, nc = int(rng.integers(1, 6)), int(rng.integers(1, 7))
        t = rng.integers(0, 4, (C, nc)).astype(np.float32)
        t[rng.random((C, nc)) < 0.15] = np.nan
        got = oracle.clip_select(t, oracle.CLIP_PER_CHANNEL)
        for k in range(C):
            fin = [c for c in range(nc) if not np.isnan(t[k, c])]
            want = min(fin, key=lambda c: (t[k, c], c)) if fin else -1
            assert got[k] == want
        got = oracle.clip_select(t, oracle.CLIP_PER_LAYER)
        sums = [float(np.sum(t[:, c].astype(np.float64))) for c in range(nc)]
        fin = [c for c in range(nc) if not np.isnan(sums[c])]
        want = min(fin, key=lambda c: (sums[c], c)) if fin else -1
        assert list(got) == [want] * C


def test_clip_single_channel_layer_and_nonfinite(oracle):
    rng = np.random.default_rng(35)
    w = rng.standard_normal((1, 50)).astype(np.float32)
    X = rng.standard_normal((9, 50)).astype(np.float32)
    a = oracle.clip_candidates(w, 20, oracle.CLIP_PER_CHANNEL)
    b = oracle.clip_candidates(w, 20, oracle.CLIP_PER_LAYER)
    assert np.array_equal(a, b)
    W = rng.standard_normal((3, 50)).astype(np.float32)
    W[1, 7] = np.inf
    c0 = oracle.clip_candidates(W, 20, oracle.CLIP_PER_CHANNEL)
    assert np.all(np.isnan(c0[1])) and np.all(np.isfinite(c0[[0, 2]]))
    e = oracle.clip_errors(X, 1, W, 4, c0).astype(np.float32)
    assert list(oracle.clip_select(e, oracle.CLIP_PER_CHANNEL))[1] == -1
    c1 = oracle.clip_candidates(W, 20, oracle.CLIP_PER_LAYER)
    assert np.all(np.isnan(c1))
    e1 = oracle.clip_errors(X, 1, W, 4, c1).astype(np.float32)
    assert list(oracle.clip_select(e1, oracle.CLIP_PER_LAYER)) == [-1, -1, -1]


# ---- Eq. 13 / Sec. 3.4: integer inference with multipoint weights ---------------------------------

def test_integer_inference_hand_example(oracle):
    g = json.load(open(os.path.join(GOLDEN, "integer_inference_hand_example.json")))
    codes = np.array(g["codes"], np.int8)
    scales = np.array(g["scales"], np.float32)
    for k in range(2):
        for i in range(2):
            assert oracle.fixed_coeff(scales[k, i], g["p"]) == g["A"][k][i]
    Y = oracle.multipoint_linear(np.array(g["X"], np.int8), codes, scales,
                                 np.array(g["npoints"], np.int32), g["p"])
    assert Y.tolist() == g["Y"]


def test_integer_inference_exact_rational(oracle):
    """Scales that are multiples of 2^-p: the result is floor(sum_i s_i (q_i . x)) exactly, checked
    with Python's rational arithmetic."""
    rng = np.random.default_rng(41)
    for p in (0, 3, 12):
        k_max, C, d, T = 3, 5, 17, 6
        codes = rng.integers(-7, 8, (k_max, C, d)).astype(np.int8)
        A = rng.integers(-2000, 2000, (C, k_max))
        scales = (A / 2.0 ** p).astype(np.float32)
        assert np.array_equal(scales.astype(np.float64) * 2.0 ** p, A)
        npts = rng.integers(0, k_max + 1, C).astype(np.int32)
        X = rng.integers(-128, 128, (T, d)).astype(np.int8)
        Y = oracle.multipoint_linear(X, codes, scales, npts, p)
        for k in range(C):
            for t in range(T):
                v = sum(Fraction(int(A[k, i]), 2 ** p) *
                        int(np.dot(codes[i, k].astype(np.int64), X[t].astype(np.int64)))
                        for i in range(npts[k]))
                assert Y[k, t] == (v.numerator // v.denominator)


def test_integer_inference_tracks_reconstruction(oracle):
    """Against Eq. 4: Y is w~^T x up to the coefficient rounding (|A/2^p - s| <= 2^-(p+1) per point
    and dot product), the floor, and the fp32 rounding of the reconstructed weights."""
    rng = np.random.default_rng(42)
    W = rng.standard_normal((12, 96)).astype(np.float32) * 0.05
    q = oracle.quantize_layer(W, 4, 32, 4)
    npts = rng.integers(1, 5, 12).astype(np.int32)
    W_hat = oracle.reconstruct(q["codes"], q["scales"], npts)
    X = rng.integers(-128, 128, (20, 96)).astype(np.int8)
    for p in (8, 16, 20):
        Y = oracle.multipoint_linear(X, q["codes"], q["scales"], npts, p).astype(np.float64)
        ref = W_hat.astype(np.float64) @ X.T.astype(np.float64)
        for k in range(12):
            acc = np.abs(q["codes"][:npts[k], k].astype(np.int64) @ X.T.astype(np.int64))
            sq = np.abs(q["scales"][k, :npts[k], None].astype(np.float64) *
                        q["codes"][:npts[k], k].astype(np.float64))
            bound = (0.5 * acc.sum(axis=0) / 2.0 ** p + 1 +
                     npts[k] * 2.0 ** -23 * np.abs(X.astype(np.float64)) @ sq.sum(axis=0))
            assert np.all(np.abs(Y[k] - ref[k]) <= bound)


def test_integer_inference_edges(oracle):
    codes = np.full((2, 1, 4), 127, np.int8)
    X = np.full((1, 4), 127, np.int8)
    big = np.array([[40000.0, 40000.0]], np.float32)        # 2 * 40000 * 64516 > 2^31: saturates
    assert oracle.multipoint_linear(X, codes, big, np.array([2], np.int32), 0)[0, 0] == 2 ** 31 - 1
    assert oracle.multipoint_linear(X, codes, -big, np.array([2], np.int32), 0)[0, 0] == -2 ** 31
    with pytest.raises(OverflowError):                        # 2^p s does not fit 32 bits
        oracle.multipoint_linear(X, codes, big, np.array([1], np.int32), 16)
    s = np.array([[0.5, 0.25]], np.float32)
    assert oracle.multipoint_linear(X, codes, s, np.array([0], np.int32), 4)[0, 0] == 0
    y2 = oracle.multipoint_linear(X, codes, s, np.array([2], np.int32), 4)
    assert np.array_equal(oracle.multipoint_linear(X, codes, s, np.array([9], np.int32), 4), y2)


# ---- Eq. 1 with B != 0: asymmetric (centred) sets ---------------------------------------------------

def _round_f32(v: Fraction) -> np.float32:
    """Correct rounding of an exact rational to fp32 (nearest, ties to even), by comparing with the
    two fp32 neighbours exactly."""
    f = np.float32(float(v))
    lo, hi = (np.nextafter(f, np.float32(-np.inf)), f) if Fraction(float(f)) > v else \
        (f, np.nextafter(f, np.float32(np.inf)))
    dl, dh = v - Fraction(float(lo)), Fraction(float(hi)) - v
    if dl != dh:
        return lo if dl < dh else hi
    return lo if (lo.view(np.uint32) & 1) == 0 else hi


def test_center_hand_example(oracle):
    g = json.load(open(os.path.join(GOLDEN, "center_hand_example.json")))
    W = np.array(g["W"], np.float32)
    for mode, key in ((oracle.CENTER_PER_CHANNEL, "per_channel"), (oracle.CENTER_PER_LAYER, "per_layer")):
        B, Wc = oracle.center(W, mode)
        assert B.tolist() == g[key]["B"] and Wc.tolist() == g[key]["Wc"]
    pt = g["points"]
    codes, scales = np.array(pt["codes"], np.int8), np.array(pt["scales"], np.float32)
    B = np.array(g["per_channel"]["B"], np.float32)
    npts = np.array(pt["npoints"], np.int32)
    assert oracle.reconstruct(codes, scales, npts, center=B).tolist() == pt["W_hat"]
    it = g["integer"]
    assert [oracle.fixed_coeff(b, it["p"]) for b in B] == it["A_B"]
    Y = oracle.multipoint_linear(np.array(it["X"], np.int8), codes, scales, npts, it["p"], center=B)
    assert Y.tolist() == it["Y"]


def test_center_is_the_rounded_midrange(oracle):
    """B = (max + min) / 2 correctly rounded to fp32 and W - B correctly rounded, against exact
    rational arithmetic, for ranges of very different magnitudes and offsets."""
    rng = np.random.default_rng(51)
    W = np.concatenate([rng.standard_normal((4, 33)) * 0.02 + 0.3,
                        rng.uniform(-1e-3, 5.0, (3, 33)),
                        rng.standard_normal((3, 33)) * 1e4 - 2.0]).astype(np.float32)
    B, Wc = oracle.center(W, oracle.CENTER_PER_CHANNEL)
    for k in range(W.shape[0]):
        mid = (Fraction(float(W[k].max())) + Fraction(float(W[k].min()))) / 2
        assert B[k] == _round_f32(mid)
        for j in range(0, 33, 4):
            assert Wc[k, j] == _round_f32(Fraction(float(W[k, j])) - Fraction(float(B[k])))
    Bl, Wl = oracle.center(W, oracle.CENTER_PER_LAYER)
    assert np.all(Bl == _round_f32((Fraction(float(W.max())) + Fraction(float(W.min()))) / 2))
    # per layer equals per channel on the layer flattened to one channel
    B1, W1 = oracle.center(W.reshape(1, -1), oracle.CENTER_PER_CHANNEL)
    assert np.all(Bl == B1[0]) and np.array_equal(Wl.reshape(1, -1), W1)


def test_center_symmetric_range_is_the_symmetric_method(oracle):
    """A channel with max = -min has B = 0: centring changes nothing, so the greedy points and the
    reconstruction equal the symmetric method's."""
    rng = np.random.default_rng(52)
    W = rng.standard_normal((6, 40)).astype(np.float32)
    W[:, 0] = np.abs(W).max(axis=1)
    W[:, 1] = -W[:, 0]
    B, Wc = oracle.center(W, oracle.CENTER_PER_CHANNEL)
    assert np.all(B == 0) and np.array_equal(Wc, W)
    q0, q1 = oracle.quantize_layer(W, 4, 32, 3), oracle.quantize_layer(Wc, 4, 32, 3)
    assert np.array_equal(q0["codes"], q1["codes"]) and np.array_equal(q0["scales"], q1["scales"])
    n = np.full(6, 2, np.int32)
    assert np.array_equal(oracle.reconstruct(q0["codes"], q0["scales"], n),
                          oracle.reconstruct(q1["codes"], q1["scales"], n, center=B))


def test_center_affine_lattice_is_exact(oracle):
    """w = B0 + s0 q with q covering -Qmax..Qmax (dyadic B0, s0): the centre is B0, the centred
    weights are s0 q, one greedy point on the full-range grid scale reproduces w exactly."""
    rng = np.random.default_rng(53)
    for bits in (3, 4):
        qm = 2 ** (bits - 1) - 1
        q = rng.integers(-qm, qm + 1, (5, 24))
        q[:, 0], q[:, 1] = qm, -qm
        B0 = np.array([0.75, -3.5, 1024.0, 0.0078125, -0.5], np.float32)
        s0 = np.array([0.125, 0.5, 2.0, 2.0 ** -12, 0.25], np.float32)
        W = (B0[:, None] + s0[:, None] * q).astype(np.float32)
        B, Wc = oracle.center(W, oracle.CENTER_PER_CHANNEL)
        assert np.array_equal(B, B0) and np.array_equal(Wc, (s0[:, None] * q).astype(np.float32))
        out = oracle.quantize_layer(Wc, bits, 4, 1)
        What = oracle.reconstruct(out["codes"], out["scales"], np.ones(5, np.int32), center=B)
        assert np.array_equal(What, W)


def test_center_nonfinite(oracle):
    W = np.random.default_rng(54).standard_normal((3, 10)).astype(np.float32)
    W[1, 4] = np.nan
    B, _ = oracle.center(W, oracle.CENTER_PER_CHANNEL)
    assert np.isnan(B[1]) and np.all(np.isfinite(B[[0, 2]]))
    Bl, _ = oracle.center(W, oracle.CENTER_PER_LAYER)
    assert np.all(np.isnan(Bl))


def test_integer_inference_with_center_exact(oracle):
    """Dyadic scales and centres: Y = floor(B sum(x) + sum_i s_i (q_i . x)) exactly (rational
    arithmetic); with no points, Y = floor(B sum(x))."""
    rng = np.random.default_rng(55)
    for p in (0, 5, 14):
        k_max, C, d, T = 3, 6, 19, 5
        codes = rng.integers(-7, 8, (k_max, C, d)).astype(np.int8)
        A = rng.integers(-3000, 3000, (C, k_max))
        AB = rng.integers(-5000, 5000, C)
        scales = (A / 2.0 ** p).astype(np.float32)
        B = (AB / 2.0 ** p).astype(np.float32)
        npts = rng.integers(0, k_max + 1, C).astype(np.int32)
        npts[0] = 0
        X = rng.integers(-128, 128, (T, d)).astype(np.int8)
        Y = oracle.multipoint_linear(X, codes, scales, npts, p, center=B)
        for k in range(C):
            for t in range(T):
                xs = int(X[t].astype(np.int64).sum())
                v = Fraction(int(AB[k]), 2 ** p) * xs + sum(
                    Fraction(int(A[k, i]), 2 ** p) *
                    int(np.dot(codes[i, k].astype(np.int64), X[t].astype(np.int64)))
                    for i in range(npts[k]))
                assert Y[k, t] == (v.numerator // v.denominator)


# --- The adaptive grid of Eq. 10 (Definition 1) -------------------------------------------------

def _gap_pairs(t):
    """Definition 1 by its pairs: half the smallest ||t_i| - |t_j|| over pairs of distinct
    magnitudes (the |t_i| != |t_j| reading), inf if there is no such pair."""
    a = np.abs(np.asarray(t, np.float64))
    best = np.inf
    for i in range(a.size):
        for j in range(a.size):
            if a[i] != a[j]:
                best = min(best, abs(a[i] - a[j]) / 2.0)
    return best


def test_adaptive_grid_hand_example(oracle):
    """Definition 1 and Eq. 10 on examples worked by hand (tests/golden)."""
    ex = json.load(open(os.path.join(GOLDEN, "adaptive_grid_hand_example.json")))
    for case in ex["minimal_gap"]:
        want = np.inf if case["delta"] == "inf" else case["delta"]
        assert oracle.minimal_gap(np.asarray(case["t"], np.float32)) == want
    g = ex["greedy"]
    out = oracle.quantize_adaptive(np.asarray([g["w"]], np.float32), g["bits"], g["k_max"], g["eta"])
    np.testing.assert_array_equal(out["scales"][0], np.asarray(g["scales"], np.float32))
    np.testing.assert_array_equal(out["codes"][:, 0, :], np.asarray(g["codes"], np.int8))
    np.testing.assert_array_equal(out["resid_sq"][0], np.asarray(g["resid_sq"]))
    np.testing.assert_array_equal(out["gamma"][0], np.asarray(g["gamma"]))
    np.testing.assert_array_equal(out["ncand"][0], np.asarray(g["ncand"]))


def test_minimal_gap_against_pairs(oracle):
    """The oracle's sorted-magnitude minimal gap equals Definition 1 evaluated pair by pair, on
    vectors with repeated magnitudes, sign flips and zeros."""
    rng = np.random.default_rng(17)
    for trial in range(200):
        d = int(rng.integers(1, 12))
        t = np.round(rng.standard_normal(d) * 8) / 8          # repeats are common
        t[rng.random(d) < 0.3] *= -1
        t = t.astype(np.float32)
        assert oracle.minimal_gap(t) == _gap_pairs(t)


def _piecewise_grid_minimum(r, bits, eta):
    """The smallest objective of Eq. 9 over the grid of Eq. 10, found without enumerating the grid:
    between consecutive code-change points s = |r_j| / (L - 1/2) the codes are constant and the
    objective is the quadratic ||r||^2 - 2 s P + s^2 N, so only the grid points nearest its
    minimiser (and the interval ends) can win.  Those few points are evaluated by the definition.
    Also returns the continuous minimum over all s > 0 (a lower bound for any grid)."""
    qmax = (1 << (bits - 1)) - 1
    r = np.asarray(r, np.float32)
    a = np.abs(r.astype(np.float64))
    delta = _gap_pairs(r)
    gamma = eta if not np.isfinite(delta) else min(delta / qmax, eta)
    R2 = float(np.sum(r.astype(np.float64) ** 2))
    M = int(np.floor(2 * qmax * np.sqrt(R2) / gamma))

    def scale(m):
        return np.float32((m * gamma) / qmax)

    def objective(s):
        q = np.clip(np.rint(r / np.float32(s)), -qmax, qmax)
        return float(np.sum((r.astype(np.float64) - np.float64(s) * q) ** 2))

    cuts = sorted({float(x) / (L - 0.5) for x in a[a > 0] for L in range(1, qmax + 1)})
    edges = [0.0] + cuts + [np.inf]
    best, cont = np.inf, np.inf
    for lo, hi in zip(edges[:-1], edges[1:]):
        inside = (lo + hi) / 2 if np.isfinite(hi) else 2 * lo + 1
        c = np.minimum(qmax, np.rint(a / inside))
        N, P = float(np.sum(c * c)), float(np.sum(a * c))
        target = P / N if N > 0 else inside
        cont = min(cont, R2 - 2 * min(max(target, lo), hi if np.isfinite(hi) else target) * P +
                   min(max(target, lo), hi if np.isfinite(hi) else target) ** 2 * N)
        m_lo = max(1, int(np.floor(lo * qmax / gamma)))
        m_hi = M if not np.isfinite(hi) else min(M, int(np.ceil(hi * qmax / gamma)))
        if m_lo > m_hi:
            continue
        m_t = min(max(int(round(target * qmax / gamma)), m_lo), m_hi)
        for m in {m_lo, m_lo + 1, m_t - 1, m_t, m_t + 1, m_hi - 1, m_hi}:
            if 1 <= m <= M:
                best = min(best, objective(scale(m)))
    return best, cont


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_adaptive_step_against_piecewise_search(oracle, bits):
    """The first greedy step over the grid of Eq. 10 reaches the smallest grid objective, found by
    the piecewise-quadratic analysis above instead of enumeration, and never beats the continuous
    optimum over all scales."""
    rng = np.random.default_rng(100 + bits)
    for trial in range(40):
        d = int(rng.integers(1, 7))
        w = (rng.standard_normal(d) * rng.choice([0.05, 1.0, 20.0])).astype(np.float32)
        out = oracle.quantize_adaptive(w[None, :], bits, 1, max_candidates=10 ** 8)
        grid_best, cont = _piecewise_grid_minimum(w, bits, oracle.ETA)
        assert out["best"][0, 0] == pytest.approx(grid_best, rel=1e-12, abs=1e-300)
        assert out["best"][0, 0] >= cont * (1 - 1e-9) - 1e-30


def test_adaptive_grid_decay_theorem1(oracle):
    """Theorem 1 under the grid of Eq. 10 (b = 2, eta = 2^-10): the residual energy never grows and
    falls by orders of magnitude within a few points, down to the eta floor."""
    W = wlm.random_weights(6, 12, 23, "normal")
    out = oracle.quantize_adaptive(W, 2, 8, max_candidates=10 ** 8)
    rs = out["resid_sq"]
    assert np.all(rs[:, 1:] <= rs[:, :-1])
    prev, nxt = rs[:, :-1], rs[:, 1:]
    assert np.all(nxt[prev > 0] < 0.5 * prev[prev > 0])   # a fixed fraction removed per point
    assert np.all(rs[:, 6] < 5e-4 * rs[:, 0])


def test_adaptive_refusal_marking(oracle):
    """A step whose grid exceeds the cap is refused: ValueError by default; with refuse="mark" its
    scale and the later ones NaN, codes 0, ncand -1 then 0, while the steps before it are kept."""
    w = np.asarray([[1.0, 0.5]], np.float32)             # grids of 2289 and 724 candidates
    with pytest.raises(ValueError):
        oracle.quantize_adaptive(w, 2, 3, max_candidates=1000)
    o = oracle.quantize_adaptive(w, 2, 3, max_candidates=1000, refuse="mark")
    np.testing.assert_array_equal(o["ncand"][0], [-1, 0, 0])
    assert np.all(np.isnan(o["scales"][0])) and np.all(o["codes"] == 0)
    assert o["resid_sq"][0, 0] == 1.25 and np.all(np.isnan(o["resid_sq"][0, 1:]))
    o = oracle.quantize_adaptive(w, 2, 3, max_candidates=2289, refuse="mark")
    np.testing.assert_array_equal(o["ncand"][0], [2289, 724, 0])
    np.testing.assert_array_equal(o["scales"][0], np.asarray([0.75, 0.25, 0.0], np.float32))


def test_adaptive_piecewise_equals_enumeration(oracle):
    """The piecewise search of the grid of Eq. 10 (code-change points by binary search, the
    objective's quadratic form to bound where its minimum can be, the definition to settle it)
    takes every decision of the enumeration: random short channels of every kind, and grids fine
    enough that neighbouring points share an fp32 scale."""
    rng = np.random.default_rng(31)
    cases = []
    for _ in range(150):
        d = int(rng.integers(1, 10))
        w = [rng.standard_normal(d), np.round(rng.standard_normal(d) * 4) / 4,
             rng.standard_normal(d) * 1e-6, rng.laplace(size=d) * 30][int(rng.integers(0, 4))]
        cases.append((w, int(rng.choice([2, 3, 4, 6, 8])), float(rng.choice([2.0 ** -10, 1e-3, 1.0])),
                      int(rng.integers(1, 4))))
    for _ in range(3):                                   # scales repeat near the top of the grid
        cases.append((rng.standard_normal(2) * 0.6, 2, 2.0 ** -24, 1))
    for w, bits, eta, k_max in cases:
        w = np.asarray(w, np.float32)[None, :]
        a = oracle.quantize_adaptive(w, bits, k_max, eta, max_candidates=6 * 10 ** 7, refuse="mark")
        b = oracle.quantize_adaptive(w, bits, k_max, eta, max_candidates=6 * 10 ** 7, refuse="mark",
                                     piecewise=True)
        np.testing.assert_array_equal(a["codes"], b["codes"])
        np.testing.assert_array_equal(a["scales"], b["scales"])
        np.testing.assert_array_equal(a["resid_sq"], b["resid_sq"])
        np.testing.assert_array_equal(a["ncand"], b["ncand"])
        np.testing.assert_array_equal(a["best"], b["best"])


@pytest.mark.parametrize("bits,d,seed", [(2, 4, 1), (3, 3, 2), (4, 3, 3)])
def test_objective_is_the_best_code_vector(oracle, bits, d, seed):
    """Eq. 9 at one scale (oracle.objective): its value is the smallest ||r - s q||^2 over every
    code vector q in {-Qmax..Qmax}^d (exhaustive, exact rationals), and its codes attain it; an
    r exactly on the lattice s Z gives 0 and those integers."""
    qmax = 2 ** (bits - 1) - 1
    rng = np.random.default_rng(seed)
    for _ in range(20):
        r = rng.standard_normal(d).astype(np.float32)
        s = np.float32(abs(rng.standard_normal()) * 0.7 + 0.05)
        E, q = oracle.objective(r, bits, s)
        best = min(sum((Fraction(float(x)) - Fraction(float(s)) * c) ** 2 for x, c in zip(r, qq))
                   for qq in itertools.product(range(-qmax, qmax + 1), repeat=d))
        got = sum((Fraction(float(x)) - Fraction(float(s)) * int(c)) ** 2 for x, c in zip(r, q))
        assert got == best
        assert abs(E - float(best)) <= 1e-12 * max(1.0, float(best))
    s = np.float32(0.375)
    ints = np.array([3, -1, 0, 2][:d], np.int64).clip(-qmax, qmax)
    E, q = oracle.objective((ints * s).astype(np.float32), bits, s)
    assert E == 0.0 and np.array_equal(q, ints)
