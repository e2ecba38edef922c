"""CPU oracle for multipoint quantization (arXiv 2002.09049) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm may
import this package.  The product path (``paper_2002_09049_gb300``) never imports, links or runs it,
and the two share no code: this package compiles ``mpq_oracle.c`` with the host C compiler and calls
it through ctypes on numpy arrays.

Each wrapper names the passage of the paper it follows; the C file states every reading of the text.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mpq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libmpq_oracle.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-std=c99", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (gcc/cc).  Returns the library path."""
    with _lock:
        if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        os.makedirs(_BUILD, exist_ok=True)
        cc = os.environ.get("CC", "cc")
        tmp = _LIB + f".{os.getpid()}.tmp"
        subprocess.run([cc, *CFLAGS, _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        L = ctypes.c_long
        D = ctypes.c_double
        lib.mpqo_candidate_errors.argtypes = [P, I, I, I, P, P, P]
        lib.mpqo_candidate_errors.restype = None
        lib.mpqo_quantize_layer.argtypes = [P, I, I, I, I, P, I, P, P, P, P, P, P, P, I, I, P]
        lib.mpqo_quantize_layer.restype = None
        lib.mpqo_output_error.argtypes = [P, I, I, P, P, P, I, I, I, P, I, I, P]
        lib.mpqo_output_error.restype = None
        lib.mpqo_allocate_budget.argtypes = [P, I, I, D, P]
        lib.mpqo_allocate_budget.restype = L
        lib.mpqo_allocate_threshold.argtypes = [P, I, I, D, P]
        lib.mpqo_allocate_threshold.restype = L
        lib.mpqo_reconstruct.argtypes = [P, P, P, P, I, I, I, P]
        lib.mpqo_center.argtypes = [P, I, I, I, P, P]
        lib.mpqo_center.restype = None
        lib.mpqo_reconstruct.restype = None
        lib.mpqo_clip_candidates.argtypes = [P, I, I, I, I, P]
        lib.mpqo_clip_candidates.restype = None
        lib.mpqo_clip_errors.argtypes = [P, I, I, P, I, I, I, I, P, P, I, I, P]
        lib.mpqo_clip_errors.restype = None
        lib.mpqo_clip_select.argtypes = [P, I, I, I, P]
        lib.mpqo_clip_select.restype = None
        lib.mpqo_fixed_coeff.argtypes = [ctypes.c_float, I, P]
        lib.mpqo_fixed_coeff.restype = ctypes.c_longlong
        lib.mpqo_multipoint_linear.argtypes = [P, I, P, P, P, P, I, I, I, I, P, I, I]
        lib.mpqo_multipoint_linear.restype = I
        lib.mpqo_minimal_gap.argtypes = [P, I, P]
        lib.mpqo_minimal_gap.restype = D
        lib.mpqo_quantize_channel_adaptive.argtypes = [P, I, I, I, D, L, P, P, P, P, P, P, P, P, P, I,
                                                       P]
        lib.mpqo_quantize_channel_adaptive.restype = I
        lib.mpqo_objective.argtypes = [P, I, I, ctypes.c_float, P]
        lib.mpqo_objective.restype = D
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _ranges(C: int, threads: int):
    threads = max(1, min(threads, C))
    step = (C + threads - 1) // threads
    return [(c0, min(C, c0 + step)) for c0 in range(0, C, step)]


def candidate_errors(r, bits: int, G: int, grid_frac=None):
    """Eq. 9 objective ||r - s_g [r/s_g]_Q||^2 for every grid point g (double), and s_g (fp32)."""
    lib = _load()
    r = _c(r, np.float32)
    gf = None if grid_frac is None else _c(grid_frac, np.float32)
    E = np.empty(G, np.float64)
    s = np.empty(G, np.float32)
    lib.mpqo_candidate_errors(_p(r), r.size, bits, G, _p(gf), _p(E), _p(s))
    return E, s


def minimal_gap(t) -> float:
    """Definition 1: half the smallest difference between two distinct element magnitudes of t
    (the pair condition read as |t_i| != |t_j|); inf with fewer than two distinct magnitudes."""
    lib = _load()
    t = _c(t, np.float32).ravel()
    work = np.empty(max(1, t.size), np.float64)
    return float(lib.mpqo_minimal_gap(_p(t), t.size, _p(work)))


ETA = 2.0 ** -10   # the maximal grid step of the paper's experiments (Sec. 5)


def quantize_adaptive(W, bits: int, k_max: int, eta: float = ETA, max_candidates: int = 10 ** 7,
                      refuse: str = "raise", piecewise: bool = False):
    """Algorithm 1 with the adaptive grid of Eq. 10 (Definition 1) for every channel of W (C x d):
    step i searches a = m * gamma, m = 1..floor(2 Qmax ||r_i|| / gamma), gamma = min(Delta_{r_i} /
    Qmax, eta), as fp32 point scales s = a / Qmax.  A plain enumeration, for small channels: a step
    whose grid would exceed ``max_candidates`` is refused -- ValueError, or with refuse="mark" its
    scale and the later ones NaN, codes 0, ncand -1 for it and 0 after.  piecewise=True takes the
    same decisions without enumerating the grid (code-change points by binary search, the
    objective's quadratic form to bound where its minimum can be, the definition to settle it),
    for grids too large to enumerate; ``second`` is NaN then.

    Returns a dict with codes [k_max][C][d] int8, scales [C][k_max] fp32, resid_sq [C][k_max+1],
    gamma [C][k_max] (the a-grid step of each step), ncand [C][k_max], best/second [C][k_max],
    rin [k_max][C][d] (the residual each step starts from)."""
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    out = dict(codes=np.zeros((k_max, C, d), np.int8), scales=np.zeros((C, k_max), np.float32),
               resid_sq=np.zeros((C, k_max + 1), np.float64),
               gamma=np.zeros((C, k_max), np.float64), ncand=np.zeros((C, k_max), np.int64),
               best=np.zeros((C, k_max), np.float64), second=np.zeros((C, k_max), np.float64),
               rin=np.zeros((k_max, C, d), np.float32))
    codes = np.zeros((k_max, d), np.int8)
    rin = np.zeros((k_max, d), np.float32)
    r = np.empty(d, np.float32)
    work = np.empty(d, np.float64)
    for k in range(C):
        st = lib.mpqo_quantize_channel_adaptive(
            _p(W[k]), d, bits, k_max, float(eta), int(max_candidates), _p(codes),
            _p(out["scales"][k]), _p(out["resid_sq"][k]), _p(out["gamma"][k]), _p(out["ncand"][k]),
            _p(out["best"][k]), _p(out["second"][k]), _p(r), _p(work), int(bool(piecewise)),
            _p(rin))
        if st < -1:
            raise RuntimeError(f"channel {k}: the piecewise search failed ({st})")
        if st != 0 and refuse == "raise":
            raise ValueError(f"channel {k}: the adaptive grid exceeds {max_candidates} candidates")
        out["codes"][:, k, :] = codes
        out["rin"][:, k, :] = rin
    return out


def objective(r, bits: int, s: float):
    """Eq. 9 at one fp32 scale by its definition: (||r - s [r/s]_Q||^2 in double, the codes)."""
    lib = _load()
    r = _c(r, np.float32).ravel()
    q = np.zeros(r.size, np.int8)
    E = lib.mpqo_objective(_p(r), r.size, bits, ctypes.c_float(np.float32(s)), _p(q))
    return float(E), q


def quantize_layer(W, bits: int, G: int, k_max: int, grid_frac=None, channels=None,
                   want_residuals: bool = True, threads: int = 1):
    """Algorithm 1 (Eq. 7-9) for every channel of W (C x d, fp32), run to k_max points.

    Returns a dict with codes [k_max][C][d] int8, scales [C][k_max] fp32, resid_sq [C][k_max+1]
    float64, residuals [k_max][C][d] fp32 (or None), gstar/best/second [C][k_max].
    ``channels`` = (c0, c1) restricts the work to a channel range (other rows stay zero).
    """
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    gf = None if grid_frac is None else _c(grid_frac, np.float32)
    out = dict(
        codes=np.zeros((k_max, C, d), np.int8),
        scales=np.zeros((C, k_max), np.float32),
        resid_sq=np.zeros((C, k_max + 1), np.float64),
        residuals=np.zeros((k_max, C, d), np.float32) if want_residuals else None,
        gstar=np.zeros((C, k_max), np.int32),
        best=np.zeros((C, k_max), np.float64),
        second=np.zeros((C, k_max), np.float64),
    )
    c0, c1 = channels if channels is not None else (0, C)

    def run(rng):
        work = np.empty(d, np.float32)
        lib.mpqo_quantize_layer(_p(W), C, d, bits, G, _p(gf), k_max, _p(out["codes"]),
                                _p(out["scales"]), _p(out["resid_sq"]), _p(out["residuals"]),
                                _p(out["gstar"]), _p(out["best"]), _p(out["second"]), rng[0], rng[1],
                                _p(work))

    _parallel(run, [(a + c0, b + c0) for a, b in _ranges(c1 - c0, threads)], threads)
    return out


def output_error(X, groups: int, W, codes, scales, k_max: int, channels=None, threads: int = 1):
    """Eq. 11 for n = 0..k_max points: err[k][n] = mean_t (x_t . r_{k,n+1})^2, in double.

    groups = 1: X is N x d (shared); groups = C: X is C x N x d (one block per channel).
    """
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    X = _c(X, np.float32)
    N = X.shape[-2]
    codes = _c(codes, np.int8)
    scales = _c(scales, np.float32)
    err = np.zeros((C, k_max + 1), np.float64)
    c0, c1 = channels if channels is not None else (0, C)

    def run(rng):
        work = np.empty(d, np.float32)
        lib.mpqo_output_error(_p(X), N, groups, _p(W), _p(codes), _p(scales), C, d, k_max,
                              _p(err), rng[0], rng[1], _p(work))

    _parallel(run, [(a + c0, b + c0) for a, b in _ranges(c1 - c0, threads)], threads)
    return err


def allocate_budget(err32, k_max: int, beta: float):
    """Budget reading of Algorithm 2: sequential marginal-gain loop on the fp32 error table."""
    lib = _load()
    err32 = _c(err32, np.float32)
    C = err32.shape[0]
    n = np.zeros(C, np.int32)
    used = lib.mpqo_allocate_budget(_p(err32), C, k_max, float(beta), _p(n))
    return n, int(used)


def allocate_threshold(err32, k_max: int, eps: float):
    """Algorithm 2: smallest n with e(n) < eps, else k_max."""
    lib = _load()
    err32 = _c(err32, np.float32)
    C = err32.shape[0]
    n = np.zeros(C, np.int32)
    used = lib.mpqo_allocate_threshold(_p(err32), C, k_max, float(eps), _p(n))
    return n, int(used)


def reconstruct(codes, scales, npoints, center=None):
    """Eq. 4: w~_k = B_k + sum_{i<=n_k} s_{k,i} q_{k,i} (fmaf chain from the centre B_k, or 0)."""
    lib = _load()
    codes = _c(codes, np.int8)
    scales = _c(scales, np.float32)
    npoints = _c(npoints, np.int32)
    k_max, C, d = codes.shape
    cen = None if center is None else _c(center, np.float32)
    W_hat = np.zeros((C, d), np.float32)
    lib.mpqo_reconstruct(_p(codes), _p(scales), _p(npoints), None if cen is None else _p(cen),
                         C, d, k_max, _p(W_hat))
    return W_hat


CENTER_PER_CHANNEL = 0
CENTER_PER_LAYER = 1


def center(W, mode: int):
    """Eq. 1 with B != 0: the centre B per channel (mode 0) or per layer (mode 1) = the midpoint of
    the weights' range in fp32, and the centred weights W - B (fp32)."""
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    B = np.zeros(C, np.float32)
    Wc = np.zeros((C, d), np.float32)
    lib.mpqo_center(_p(W), C, d, mode, _p(B), _p(Wc))
    return B, Wc


CLIP_PER_CHANNEL = 0
CLIP_PER_LAYER = 1


def clip_candidates(W, n_cand: int, mode: int):
    """Eq. 12's candidate clipping factors K_c = (c+1)/n_cand * max|w| (per channel or per layer)."""
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    clip = np.zeros((C, n_cand), np.float32)
    lib.mpqo_clip_candidates(_p(W), C, d, n_cand, mode, _p(clip))
    return clip


def clip_errors(X, groups: int, W, bits: int, clip, channels=None, threads: int = 1):
    """Eq. 12's objective: output error (Eq. 11 form) of every candidate clipping factor, in double."""
    lib = _load()
    W = _c(W, np.float32)
    C, d = W.shape
    X = _c(X, np.float32)
    N = X.shape[-2]
    clip = _c(clip, np.float32)
    n_cand = clip.shape[1]
    err = np.zeros((C, n_cand), np.float64)
    c0, c1 = channels if channels is not None else (0, C)

    def run(rng):
        work = np.empty(d, np.float32)
        lib.mpqo_clip_errors(_p(X), N, groups, _p(W), C, d, bits, n_cand, _p(clip), _p(err),
                             rng[0], rng[1], _p(work))

    _parallel(run, [(a + c0, b + c0) for a, b in _ranges(c1 - c0, threads)], threads)
    return err


def clip_select(err32, mode: int):
    """Eq. 12's argmin on an fp32 error table: per channel, or per layer (sum over channels)."""
    lib = _load()
    err32 = _c(err32, np.float32)
    C, n_cand = err32.shape
    best = np.zeros(C, np.int32)
    lib.mpqo_clip_select(_p(err32), C, n_cand, mode, _p(best))
    return best


def fixed_coeff(s: float, p: int):
    """Eq. 13: A = rint(2^p s) as an int; None when it does not fit 32 bits."""
    lib = _load()
    ok = ctypes.c_int(1)
    a = lib.mpqo_fixed_coeff(float(s), p, ctypes.byref(ok))
    return int(a) if ok.value else None


def multipoint_linear(X, codes, scales, npoints, p: int, channels=None, threads: int = 1,
                      center=None):
    """Sec. 3.4 steps 1-3: Y [C][T] int32 = sat32(floor(sum_i A_i (q_i . x_t) / 2^p)), exact; with
    a centre B (asymmetric set), A_B (sum_j x_tj) joins the sum, A_B = rint(2^p B)."""
    lib = _load()
    cen = None if center is None else _c(center, np.float32)
    X = _c(X, np.int8)
    codes = _c(codes, np.int8)
    scales = _c(scales, np.float32)
    npoints = _c(npoints, np.int32)
    T, d = X.shape
    k_max, C, _ = codes.shape
    Y = np.zeros((C, T), np.int32)
    c0, c1 = channels if channels is not None else (0, C)
    bad = []

    def run(rng):
        if lib.mpqo_multipoint_linear(_p(X), T, _p(codes), _p(scales), _p(npoints),
                                      None if cen is None else _p(cen), C, d, k_max, p, _p(Y),
                                      rng[0], rng[1]):
            bad.append(rng)

    _parallel(run, [(a + c0, b + c0) for a, b in _ranges(c1 - c0, threads)], threads)
    if bad:
        raise OverflowError("a coefficient 2^p * s does not fit 32 bits")
    return Y


def _parallel(fn, ranges, threads):
    """Channels are independent: ranges run on a thread pool (ctypes drops the GIL in C calls)."""
    if threads <= 1 or len(ranges) == 1:
        for rng in ranges:
            fn(rng)
        return
    with ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(fn, ranges))
