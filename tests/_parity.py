"""Comparison rules between the CUDA path and the oracle (used by the gpu tests, smoke, bench).

Codes and scales must be bit-exact.  The one allowed exception is a near tie of the scale search:
the oracle's error at the candidate the GPU chose is within 1e-6 relative of the oracle's best.
After such a step the channel's later steps start from a different residual and are excluded from
value comparison ("diverged after near tie").  Float values (resid_sq, err) must agree within
1e-5 relative; residuals and reconstructions, which follow the same fp32 recursion, bit-exactly.
"""
from __future__ import annotations

import numpy as np

NEAR_TIE_RTOL = 1e-6
VALUE_RTOL = 1e-5


def _grid(m, qmax, G, grid_frac):
    smax = np.float32(m) / np.float32(qmax)
    f = (np.arange(1, G + 1, dtype=np.float32) / np.float32(G)) if grid_frac is None else \
        np.asarray(grid_frac, np.float32)
    return (f * smax).astype(np.float32)


def _same_scale(a, b):
    """Bit-identical fp32 scales; any two NaNs (a channel with a non-finite weight) match."""
    if np.isnan(a) and np.isnan(b):
        return True
    return a.tobytes() == b.tobytes()


def compare_quantize(W, gpu: dict, orc: dict, bits: int, G: int, k_max: int, grid_frac=None,
                     oracle=None, channels=None):
    """Returns a report dict; raises AssertionError on any non-near-tie mismatch.

    gpu: codes [k_max][C][d], scales [C][k_max], resid_sq [C][k_max+1] (and optionally residuals).
    orc: the oracle's quantize_layer output.  channels: iterable of channel indices to check."""
    qmax = 2 ** (bits - 1) - 1
    C, d = W.shape
    chans = range(C) if channels is None else channels
    near_ties = 0
    diverged_steps = 0
    checked = 0
    for k in chans:
        diverged = False
        for i in range(k_max):
            if diverged:
                diverged_steps += 1
                continue
            same_s = _same_scale(gpu["scales"][k, i], orc["scales"][k, i])
            same_q = np.array_equal(gpu["codes"][i, k], orc["codes"][i, k])
            if same_s and same_q:
                checked += 1
                if "residuals" in gpu and gpu["residuals"] is not None:
                    assert np.array_equal(gpu["residuals"][i, k], orc["residuals"][i, k],
                                          equal_nan=True), f"residual mismatch k={k} i={i}"
                continue
            # mismatch: must be a near tie of this step's scale search
            assert oracle is not None, f"mismatch at k={k} step={i} and no oracle to judge it"
            r = W[k] if i == 0 else orc["residuals"][i - 1, k]
            E, s = oracle.candidate_errors(r, bits, G, grid_frac)
            gs = np.nonzero(s == gpu["scales"][k, i])[0]
            assert gs.size > 0, f"k={k} step={i}: GPU scale {gpu['scales'][k, i]!r} not on grid"
            Eg = E[gs[0]]
            Eb = E.min()
            assert Eg <= Eb + NEAR_TIE_RTOL * Eb, (
                f"k={k} step={i}: GPU took scale {gpu['scales'][k, i]!r} with E={Eg!r}, oracle "
                f"best {orc['scales'][k, i]!r} E={Eb!r} (rel gap {(Eg - Eb) / max(Eb, 1e-300):.3e})")
            near_ties += 1
            diverged = True
        # resid_sq of the agreeing prefix
        n_ok = k_max + 1 if not diverged else None
        if n_ok is None:
            # steps before the first divergence (plus the initial norm)
            agree = 0
            for i in range(k_max):
                if _same_scale(gpu["scales"][k, i], orc["scales"][k, i]) and \
                        np.array_equal(gpu["codes"][i, k], orc["codes"][i, k]):
                    agree += 1
                else:
                    break
            n_ok = agree + 1
        if gpu.get("resid_sq") is not None:
            g = gpu["resid_sq"][k, :n_ok].astype(np.float64)
            o = orc["resid_sq"][k, :n_ok]
            finite = np.isfinite(o)
            assert np.array_equal(np.isnan(g), np.isnan(o)), f"NaN pattern of resid_sq k={k}"
            np.testing.assert_allclose(g[finite], o[finite], rtol=VALUE_RTOL, atol=1e-30,
                                       err_msg=f"resid_sq k={k}")
    return dict(near_ties=near_ties, diverged_steps=diverged_steps, checked_steps=checked)


def compare_err(gpu_err, orc_err, rtol=VALUE_RTOL):
    g = np.asarray(gpu_err, np.float64)
    o = np.asarray(orc_err, np.float64)
    assert np.array_equal(np.isnan(g), np.isnan(o))
    f = np.isfinite(o)
    rel = np.abs(g[f] - o[f]) / np.maximum(np.abs(o[f]), 1e-300)
    worst = float(rel.max()) if rel.size else 0.0
    assert worst <= rtol, f"output error max rel diff {worst:.3e} > {rtol}"
    return worst


def _on_adaptive_grid(s: np.float32, gamma: float, qmax: int, M: int) -> bool:
    """Whether s is one of the step's grid scales fl32(fl64(m gamma) / Qmax), m = 1..M."""
    if s == 0.0:
        return M >= 1 and np.float32(gamma / qmax) == 0.0
    c = float(s) * qmax / gamma
    w = int(c * 2.0 ** -21) + 4
    for m in range(max(1, int(c) - w), min(M, int(c) + w) + 1):
        if np.float32((m * gamma) / qmax) == s:
            return True
    return False


def compare_adaptive(gpu: dict, orc: dict, bits: int, oracle, channels=None):
    """The adaptive grid (Eq. 10) on the GPU against the oracle (enumeration or its piecewise
    search, both the definition's first minimiser).  Per channel and step: grid size ncand,
    scale, codes and squared residual norm bit-exact; the one exception is a near tie -- the GPU's
    scale is a grid point of that step whose codes are the definition's and whose objective is
    within 1e-6 relative of the oracle's best -- after which the channel's later steps are
    excluded.  gpu: codes [k][C][d], scales [C][k], resid_sq [C][k+1], ncand [C][k].
    Returns the number of near ties."""
    qmax = 2 ** (bits - 1) - 1
    k_max = gpu["scales"].shape[1]
    chans = range(gpu["scales"].shape[0]) if channels is None else channels
    near = 0
    for k in chans:
        assert gpu["resid_sq"][k, 0].tobytes() == np.float32(orc["resid_sq"][k, 0]).tobytes() or \
            (np.isnan(gpu["resid_sq"][k, 0]) and np.isnan(orc["resid_sq"][k, 0])), f"k={k} norm"
        for i in range(k_max):
            assert gpu["ncand"][k, i] == orc["ncand"][k, i], \
                f"k={k} step={i}: grid size {gpu['ncand'][k, i]} vs {orc['ncand'][k, i]}"
            sg, so = gpu["scales"][k, i], orc["scales"][k, i]
            same = (_same_scale(sg, so) and np.array_equal(gpu["codes"][i, k], orc["codes"][i, k]))
            if not same:
                assert not _same_scale(sg, so), f"k={k} step={i}: same scale, other codes"
                r = orc["rin"][i, k]
                E, q = oracle.objective(r, bits, sg)
                assert np.array_equal(gpu["codes"][i, k], q), f"k={k} step={i}: codes"
                assert _on_adaptive_grid(sg, float(orc["gamma"][k, i]), qmax,
                                         int(orc["ncand"][k, i])), f"k={k} step={i}: off grid"
                Eb = float(orc["best"][k, i])
                assert E <= Eb + NEAR_TIE_RTOL * abs(Eb), (
                    f"k={k} step={i}: GPU scale {sg!r} E={E!r}, oracle {so!r} E={Eb!r}")
                near += 1
                break
            r2g, r2o = gpu["resid_sq"][k, i + 1], np.float32(orc["resid_sq"][k, i + 1])
            assert r2g.tobytes() == r2o.tobytes() or (np.isnan(r2g) and np.isnan(r2o)), \
                f"k={k} step={i}: squared norm {r2g!r} vs {r2o!r}"
    return near
