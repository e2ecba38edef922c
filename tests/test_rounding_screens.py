"""Host check of the reciprocal screens the kernels use for the codes of Eq. 8.

The exact code is clamp(rint(fl(w / s)), -Qmax, Qmax) with fl the correctly rounded fp32 division.
The kernels first take q' = fl(w * inv) with inv an fp32 reciprocal of s and decide from rint(q')
unless q' lies too close to a half-integer; only then do they divide.  These tests replay that
decision in numpy's IEEE fp32 arithmetic on quotients placed next to every half-integer of the
code range (and beyond the clamp), and require that whenever a screen accepts q', its code is the
exact one:

* the signed screen (the clipping search's residual planes, the greedy search's update): unsure
  when |q' - rint(q')| >= 0.5 - 2^-20 (Qmax + 2) and |q'| < Qmax + 1; the reciprocal is fl(1/s)
  or, in the greedy search, fl(1/f_g) fl(1/smax);
* the unsigned screen on a = |w| (the greedy search's lattice events): accepted when
  0.5 - |q' - rint(q')| > 2^-20 (q' + 1).
"""
import numpy as np
import pytest

F = np.float32
REL = F(2.0 ** -20)


def exact_code(w, s, qmax):
    return np.clip(np.rint(w / s), -qmax, qmax)          # fp32 division, ties to even


def signed_screen(w, inv, qmax):
    qf = w * inv
    rq = np.rint(qf)
    qlim = F(qmax + 1)
    tband = F(0.5) - REL * (qlim + F(1))
    unsure = (np.abs(qf - rq) >= tband) & (np.abs(qf) < qlim)
    return np.clip(rq, -qmax, qmax), unsure


def unsigned_screen(a, inv, qmax):
    qf = a * inv
    rq = np.rint(qf)
    ok = (F(0.5) - np.abs(qf - rq)) > REL * (qf + F(1))
    return np.minimum(rq, F(qmax)), ok


def near_half_integers(rng, qmax, n):
    """Scales over many binades and weights whose exact quotient lies within a few ulps of
    k + 1/2 (k up to Qmax + 2, both signs), plus uniform quotients across and past the clamp."""
    s = (rng.uniform(1.0, 2.0, n) * np.exp2(rng.integers(-60, 60, n))).astype(F)
    k = rng.integers(0, qmax + 3, n).astype(np.float64)
    ulps = rng.integers(-6, 7, n).astype(np.float64)
    t = (k + 0.5) * (1.0 + ulps * 2.0 ** -24)
    t[: n // 4] = rng.uniform(0.0, qmax + 3.0, n // 4)
    sign = np.where(rng.random(n) < 0.5, -1.0, 1.0)
    w = (sign * t * s.astype(np.float64)).astype(F)
    return w, s


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_signed_screen_with_a_correct_reciprocal(bits):
    qmax = 2 ** (bits - 1) - 1
    rng = np.random.default_rng(100 + bits)
    w, s = near_half_integers(rng, qmax, 400_000)
    inv = F(1) / s
    q, unsure = signed_screen(w, inv, qmax)
    exact = exact_code(w, s, qmax)
    assert np.array_equal(q[~unsure], exact[~unsure])
    # the band is hit next to the half-integers, and uniform quotients (the first quarter) almost
    # never fall in it
    assert unsure.any() and unsure[: len(w) // 4].mean() < 1e-3


@pytest.mark.parametrize("bits", [3, 4, 8])
def test_signed_screen_with_a_product_of_reciprocals(bits):
    """The greedy search's update: inv = fl(1/f_g) * fl(1/smax), s = fl(f_g * smax)."""
    qmax = 2 ** (bits - 1) - 1
    rng = np.random.default_rng(200 + bits)
    n = 400_000
    G = 256
    f = (rng.integers(1, G + 1, n) / np.float64(G)).astype(F)     # fl((g+1)/G)
    smax = (rng.uniform(1.0, 2.0, n) * np.exp2(rng.integers(-40, 40, n))).astype(F)
    s = f * smax
    k = rng.integers(0, qmax + 3, n).astype(np.float64)
    t = (k + 0.5) * (1.0 + rng.integers(-6, 7, n) * 2.0 ** -24)
    t[: n // 4] = rng.uniform(0.0, qmax + 3.0, n // 4)
    w = (np.where(rng.random(n) < 0.5, -1.0, 1.0) * t * s.astype(np.float64)).astype(F)
    inv = (F(1) / f) * (F(1) / smax)
    q, unsure = signed_screen(w, inv, qmax)
    exact = exact_code(w, s, qmax)
    assert np.array_equal(q[~unsure], exact[~unsure])


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_unsigned_screen(bits):
    qmax = 2 ** (bits - 1) - 1
    rng = np.random.default_rng(300 + bits)
    w, s = near_half_integers(rng, qmax, 400_000)
    a = np.abs(w)
    q, ok = unsigned_screen(a, F(1) / s, qmax)
    exact = np.minimum(np.rint(a / s), F(qmax))
    assert np.array_equal(q[ok], exact[ok])


def test_screens_disagree_with_a_plain_multiply_without_the_band():
    """The band is needed: rounding the multiply's quotient alone picks a different code for
    some quotients next to a half-integer."""
    rng = np.random.default_rng(7)
    w, s = near_half_integers(rng, 7, 400_000)
    plain = np.clip(np.rint(w * (F(1) / s)), -7, 7)
    assert not np.array_equal(plain, exact_code(w, s, 7))
