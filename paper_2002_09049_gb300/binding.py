"""Thin Python binding of libmpq.so (include/mpq.h): torch tensors in, C-ABI calls out.

Every function here only checks tensor placement/shape/dtype, allocates outputs with torch when
the caller did not pass them, and forwards raw device pointers plus the current CUDA stream to the
library.  All arithmetic happens in the library's CUDA kernels; there is no CPU fallback -- if the
library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import _build

MPQ_ALLOC_BUDGET = 0
MPQ_ALLOC_THRESHOLD = 1
MPQ_CENTER_PER_CHANNEL = 0
MPQ_CENTER_PER_LAYER = 1
MPQ_CLIP_PER_CHANNEL = 0
MPQ_CLIP_PER_LAYER = 1
MPQ_NOALLOC_RANGE_WORDS = 1 << 20     # the fixed scratch of mpq_output_error_noalloc
MPQ_ADAPTIVE_MAX_THRESHOLDS = 1 << 16  # most d * Qmax of mpq_quantize_layer_adaptive
MPQ_TIMEOUT_OUTPUT_ERROR = 0x1        # timeout bits of mpq_device_status
MPQ_TIMEOUT_CLIP = 0x2
MPQ_TIMEOUT_INFERENCE = 0x4
MPQ_TIMEOUT_DRAIN = 0x100
MPQ_FAULT_BOUNDS = 0x10000            # mpq_device_status: the checked build skipped accesses
MPQ_BUILD_CHECK_BOUNDS = 0x1          # mpq_build_options: the checked build

MPQ_STATUS = {0: "MPQ_OK", 1: "MPQ_ERR_INVALID_ARG", 2: "MPQ_ERR_NONFINITE",
              3: "MPQ_ERR_UNSUPPORTED", 4: "MPQ_ERR_CUDA", 5: "MPQ_ERR_TIMEOUT",
              6: "MPQ_ERR_NOMEM", 7: "MPQ_ERR_BOUNDS"}

# name -> (argtypes, restype), in the order of include/mpq.h
_P, _I, _D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
class PackedLayout(ctypes.Structure):
    """mpq_packed_layout of include/mpq.h: the layout of a packed multipoint layer (Sec. 3.4)."""
    _fields_ = [("C", ctypes.c_int), ("d", ctypes.c_int), ("k_max", ctypes.c_int),
                ("bits", ctypes.c_int), ("p", ctypes.c_int), ("centered", ctypes.c_int),
                ("d_pad", ctypes.c_int), ("rows", ctypes.c_int), ("tiles", ctypes.c_int),
                ("off_coef", ctypes.c_size_t), ("off_chan", ctypes.c_size_t),
                ("off_point", ctypes.c_size_t), ("off_tile", ctypes.c_size_t),
                ("off_center", ctypes.c_size_t), ("off_codes", ctypes.c_size_t),
                ("bytes", ctypes.c_size_t)]


_L = ctypes.POINTER(PackedLayout)

SIGNATURES = {
    "mpq_quantize_layer": ([_P, _I, _I, _I, _I, _P, _I, _P, _P, _P, _P, _P, _P], _I),
    "mpq_quantize_layer_adaptive": ([_P, _I, _I, _I, _I, _D, ctypes.c_longlong, _P, _P, _P, _P,
                                     _P], _I),
    "mpq_output_error": ([_P, _I, _I, _P, _P, _P, _P, _I, _I, _I, _P, _P], _I),
    "mpq_output_error_noalloc": ([_P, _I, _I, _P, _P, _P, _I, _I, _I, _P, _P], _I),
    "mpq_allocate_points": ([_P, _I, _I, _I, _D, _P, _P, _P], _I),
    "mpq_allocate_points_batched": ([_I, _P, _P, _I, _I, _P, _P, _P, _P], _I),
    "mpq_reconstruct": ([_P, _P, _P, _P, _I, _I, _I, _P, _P], _I),
    "mpq_center_weights": ([_P, _I, _I, _I, _P, _P, _P], _I),
    "mpq_clip_search": ([_P, _I, _I, _P, _I, _I, _I, _I, _I, _P, _P, _P, _P], _I),
    "mpq_pack_layout": ([_P, _I, _I, _I, _I, _I, _I, _L], _I),
    "mpq_pack_points": ([_P, _P, _P, _P, _L, _P, _P], _I),
    "mpq_multipoint_linear": ([_P, _I, _L, _P, _P, _P], _I),
    "mpq_device_status": ([_P, _P], _I),
    "mpq_set_wait_limit": ([ctypes.c_longlong], _I),
    "mpq_test_withhold_copies": ([_I], _I),
    "mpq_build_options": ([], ctypes.c_uint),
    "mpq_status_string": ([_I], ctypes.c_char_p),
    "mpq_last_error": ([], ctypes.c_char_p),
    "mpq_version": ([], _I),
}

_lib = None


class MPQError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        self.status = status
        super().__init__(f"{where}: {MPQ_STATUS.get(status, status)}: {detail}")


def lib_path() -> str:
    return _build.LIB


def load(path: str | None = None):
    """Loads libmpq.so (built by __graft_entry__.build() / paper_2002_09049_gb300._build), or the
    library the MPQ_LIBRARY environment variable names (the checked build, libmpq_checked.so)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or os.environ.get("MPQ_LIBRARY") or _build.LIB
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build it with paper_2002_09049_gb300._build.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(p)
    for name, (argt, rest) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.argtypes = argt
        fn.restype = rest
    if path is None:
        _lib = lib
    return lib


def _check(status: int, where: str):
    if status != 0:
        detail = load().mpq_last_error().decode(errors="replace")
        raise MPQError(status, where, detail)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, name, dtype, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t


def mpq_quantize_layer(W, bits: int, G: int, k_max: int, grid_frac=None, codes=None,
                       scales=None, resid_sq=None, residuals=None, want_resid_sq=True,
                       rmax=None, stream=None):
    """Greedy multipoint construction (Algorithm 1) of every channel of W [C][d] fp32.

    Returns (codes [k_max][C][d] int8, scales [C][k_max] fp32, resid_sq [C][k_max+1] or None,
    residuals or None).  grid_frac: optional host sequence of G fractions in (0, 1].  rmax: an
    optional [C][k_max+1] fp32 tensor that receives max |r| of every residual vector."""
    _dev(W, "W", torch.float32)
    C, d = W.shape
    dev = W.device
    codes = codes if codes is not None else torch.empty((k_max, C, d), dtype=torch.int8, device=dev)
    scales = scales if scales is not None else torch.empty((C, k_max), dtype=torch.float32,
                                                           device=dev)
    if resid_sq is None and want_resid_sq:
        resid_sq = torch.empty((C, k_max + 1), dtype=torch.float32, device=dev)
    _dev(codes, "codes", torch.int8, (k_max, C, d))
    _dev(scales, "scales", torch.float32, (C, k_max))
    if resid_sq is not None:
        _dev(resid_sq, "resid_sq", torch.float32, (C, k_max + 1))
    if residuals is not None:
        _dev(residuals, "residuals", torch.float32, (k_max, C, d))
    if rmax is not None:
        _dev(rmax, "rmax", torch.float32, (C, k_max + 1))
    gf = None
    if grid_frac is not None:
        gf_list = [float(x) for x in grid_frac]
        if len(gf_list) != G:
            raise ValueError("grid_frac must have G entries")
        gf = (ctypes.c_float * G)(*gf_list)
    st = load().mpq_quantize_layer(_ptr(W), C, d, bits, G, gf, k_max, _ptr(codes), _ptr(scales),
                                   _ptr(resid_sq), _ptr(residuals), _ptr(rmax), _stream(stream))
    _check(st, "mpq_quantize_layer")
    return codes, scales, resid_sq, residuals


ETA = 2.0 ** -10   # the largest grid step of the paper's experiments


def mpq_quantize_layer_adaptive(W, bits: int, k_max: int, eta: float = ETA,
                                max_cand: int = 10 ** 7, codes=None, scales=None, resid_sq=None,
                                ncand=None, stream=None):
    """Algorithm 1 with the adaptive grid of Eq. 10 (Definition 1), d * Qmax <=
    MPQ_ADAPTIVE_MAX_THRESHOLDS.  Returns (codes [k_max][C][d] int8, scales [C][k_max] fp32,
    resid_sq [C][k_max+1] fp32, ncand [C][k_max] int64: each step's grid size, -1 if refused)."""
    _dev(W, "W", torch.float32)
    C, d = W.shape
    dev = W.device
    codes = codes if codes is not None else torch.empty((k_max, C, d), dtype=torch.int8, device=dev)
    scales = scales if scales is not None else torch.empty((C, k_max), dtype=torch.float32,
                                                           device=dev)
    resid_sq = resid_sq if resid_sq is not None else torch.empty((C, k_max + 1),
                                                                 dtype=torch.float32, device=dev)
    ncand = ncand if ncand is not None else torch.empty((C, k_max), dtype=torch.int64, device=dev)
    _dev(codes, "codes", torch.int8, (k_max, C, d))
    _dev(scales, "scales", torch.float32, (C, k_max))
    _dev(resid_sq, "resid_sq", torch.float32, (C, k_max + 1))
    _dev(ncand, "ncand", torch.int64, (C, k_max))
    st = load().mpq_quantize_layer_adaptive(_ptr(W), C, d, bits, k_max, float(eta), int(max_cand),
                                            _ptr(codes), _ptr(scales), _ptr(resid_sq),
                                            _ptr(ncand), _stream(stream))
    _check(st, "mpq_quantize_layer_adaptive")
    return codes, scales, resid_sq, ncand


def _output_error(entry, X, W, codes, scales, k_max, groups, err, stream, rmax=None):
    _dev(W, "W", torch.float32)
    C, d = W.shape
    _dev(X, "X", torch.float32)
    if groups == 1:
        if X.dim() != 2 or X.shape[1] != d:
            raise ValueError("X must be [N][d] for groups = 1")
        N = X.shape[0]
    else:
        if X.dim() != 3 or X.shape[0] != C or X.shape[2] != d:
            raise ValueError("X must be [C][N][d] for groups = C")
        N = X.shape[1]
    _dev(codes, "codes", torch.int8, (k_max, C, d))
    _dev(scales, "scales", torch.float32, (C, k_max))
    err = err if err is not None else torch.empty((C, k_max + 1), dtype=torch.float32,
                                                  device=W.device)
    _dev(err, "err", torch.float32, (C, k_max + 1))
    if entry == "mpq_output_error":
        if rmax is not None:
            _dev(rmax, "rmax", torch.float32, (C, k_max + 1))
        st = load().mpq_output_error(_ptr(X), N, groups, _ptr(W), _ptr(codes), _ptr(scales),
                                     _ptr(rmax), C, d, k_max, _ptr(err), _stream(stream))
    else:
        st = getattr(load(), entry)(_ptr(X), N, groups, _ptr(W), _ptr(codes), _ptr(scales), C,
                                    d, k_max, _ptr(err), _stream(stream))
    _check(st, entry)
    return err


def mpq_output_error(X, W, codes, scales, k_max: int, groups: int = 1, err=None, stream=None,
                     rmax=None):
    """Output error (Eq. 11) for n = 0..k_max points: err [C][k_max+1] fp32.  rmax: the greedy
    search's max |r| per residual vector, if kept (the ranges are then not measured again)."""
    return _output_error("mpq_output_error", X, W, codes, scales, k_max, groups, err, stream,
                         rmax)


def mpq_output_error_noalloc(X, W, codes, scales, k_max: int, groups: int = 1, err=None,
                             stream=None):
    """mpq_output_error through the entry point that allocates nothing (one fixed scratch buffer
    inside the library: calls must not overlap)."""
    return _output_error("mpq_output_error_noalloc", X, W, codes, scales, k_max, groups, err,
                         stream)


def mpq_clip_search(X, W, bits: int, n_cand: int = 20, mode: int = None, groups: int = 1,
                    clip=None, err=None, best=None, stream=None):
    """Output-error-driven clipping factor (Eq. 12) among n_cand candidates (c+1)/n_cand x max|w|:
    returns (clip [C][n_cand] fp32, err [C][n_cand] fp32, best [C] int32)."""
    mode = MPQ_CLIP_PER_CHANNEL if mode is None else mode
    _dev(W, "W", torch.float32)
    C, d = W.shape
    _dev(X, "X", torch.float32)
    if groups == 1:
        if X.dim() != 2 or X.shape[1] != d:
            raise ValueError("X must be [N][d] for groups = 1")
        N = X.shape[0]
    else:
        if X.dim() != 3 or X.shape[0] != C or X.shape[2] != d:
            raise ValueError("X must be [C][N][d] for groups = C")
        N = X.shape[1]
    mk = lambda dt: torch.empty((C, n_cand), dtype=dt, device=W.device)
    clip = clip if clip is not None else mk(torch.float32)
    err = err if err is not None else mk(torch.float32)
    best = best if best is not None else torch.empty((C,), dtype=torch.int32, device=W.device)
    _dev(clip, "clip", torch.float32, (C, n_cand))
    _dev(err, "err", torch.float32, (C, n_cand))
    _dev(best, "best", torch.int32, (C,))
    st = load().mpq_clip_search(_ptr(X), N, groups, _ptr(W), C, d, bits, n_cand, mode, _ptr(clip),
                                _ptr(err), _ptr(best), _stream(stream))
    _check(st, "mpq_clip_search")
    return clip, err, best


def _host_int32(a):
    import numpy as np
    if isinstance(a, torch.Tensor):
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(a, dtype=np.int32)


def mpq_pack_layout(npoints, d: int, k_max: int, bits: int, p: int,
                    centered: bool = False) -> PackedLayout:
    """Host-side layout of a packed multipoint layer (Sec. 3.4) for the point counts npoints [C]
    (centered: the layer has centres B_k of asymmetric sets)."""
    n = _host_int32(npoints)
    lay = PackedLayout()
    st = load().mpq_pack_layout(n.ctypes.data, int(n.size), d, k_max, bits, p, int(bool(centered)),
                                ctypes.byref(lay))
    _check(st, "mpq_pack_layout")
    return lay


def mpq_pack_points(codes, scales, npoints, layout: PackedLayout, packed=None, stream=None,
                    center=None):
    """Coefficients rint(2^p s) and bf16 codes of the used points, and rint(2^p B) of the centres
    when the layout is centered (offline, synchronous).  Returns the packed device buffer
    (uint8 [layout.bytes])."""
    _dev(codes, "codes", torch.int8, (layout.k_max, layout.C, layout.d))
    _dev(scales, "scales", torch.float32, (layout.C, layout.k_max))
    if center is not None:
        _dev(center, "center", torch.float32, (layout.C,))
    n = _host_int32(npoints)
    if n.size != layout.C:
        raise ValueError("npoints must have C entries")
    packed = packed if packed is not None else torch.empty((max(1, layout.bytes),), dtype=torch.uint8,
                                                           device=codes.device)
    _dev(packed, "packed", torch.uint8)
    if packed.numel() < layout.bytes:
        raise ValueError("packed buffer smaller than layout.bytes")
    st = load().mpq_pack_points(_ptr(codes), _ptr(scales), _ptr(center), n.ctypes.data,
                                ctypes.byref(layout), _ptr(packed), _stream(stream))
    _check(st, "mpq_pack_points")
    return packed


def mpq_multipoint_linear(X, layout: PackedLayout, packed, Y=None, stream=None):
    """Integer inference (Eq. 13): Y [C][T] int32 for X [T][d] int8."""
    _dev(X, "X", torch.int8)
    if X.dim() != 2 or X.shape[1] != layout.d:
        raise ValueError("X must be [T][d]")
    T = X.shape[0]
    Y = Y if Y is not None else torch.empty((layout.C, T), dtype=torch.int32, device=X.device)
    _dev(Y, "Y", torch.int32, (layout.C, T))
    st = load().mpq_multipoint_linear(_ptr(X), T, ctypes.byref(layout), _ptr(packed), _ptr(Y),
                                      _stream(stream))
    _check(st, "mpq_multipoint_linear")
    return Y


def mpq_allocate_points(err, k_max: int, mode: int = MPQ_ALLOC_BUDGET,
                        budget_or_eps: float = 1.0, npoints=None, points_used=None, stream=None):
    """Per-channel point counts (Algorithm 2, budget or threshold mode).

    Returns (npoints [C] int32, points_used [1] int32) on the device."""
    _dev(err, "err", torch.float32)
    C = err.shape[0]
    if tuple(err.shape) != (C, k_max + 1):
        raise ValueError("err must be [C][k_max+1]")
    npoints = npoints if npoints is not None else torch.empty((C,), dtype=torch.int32,
                                                              device=err.device)
    points_used = points_used if points_used is not None else torch.empty(
        (1,), dtype=torch.int32, device=err.device)
    _dev(npoints, "npoints", torch.int32, (C,))
    _dev(points_used, "points_used", torch.int32, (1,))
    st = load().mpq_allocate_points(_ptr(err), C, k_max, mode, float(budget_or_eps),
                                    _ptr(npoints), _ptr(points_used), _stream(stream))
    _check(st, "mpq_allocate_points")
    return npoints, points_used


MPQ_MAX_BATCH = 64


def mpq_allocate_points_batched(errs, k_max: int, mode: int, budgets, npoints=None,
                                points_used=None, stream=None):
    """Algorithm 2 for several layers in one launch: errs[l] is layer l's [C_l][k_max+1] fp32
    error table, budgets[l] its beta (budget mode) or eps.  Returns (npoints list, points_used
    list); pass lists of preallocated tensors to write into them instead."""
    n = len(errs)
    if n > MPQ_MAX_BATCH:
        raise ValueError(f"at most {MPQ_MAX_BATCH} layers per call")
    Cs = []
    for e in errs:
        _dev(e, "err", torch.float32)
        if e.dim() != 2 or e.shape[1] != k_max + 1:
            raise ValueError("every err must be [C][k_max+1]")
        Cs.append(e.shape[0])
    if npoints is None:
        npoints = [torch.empty((c,), dtype=torch.int32, device=e.device) for c, e in zip(Cs, errs)]
    if points_used is None:
        points_used = [torch.empty((1,), dtype=torch.int32, device=e.device) for e in errs]
    for c, t in zip(Cs, npoints):
        _dev(t, "npoints", torch.int32, (c,))
    for t in points_used:
        _dev(t, "points_used", torch.int32, (1,))
    P = ctypes.c_void_p * max(1, n)
    st = load().mpq_allocate_points_batched(
        n, P(*[e.data_ptr() for e in errs]), (ctypes.c_int * max(1, n))(*Cs), k_max, mode,
        (ctypes.c_double * max(1, n))(*[float(b) for b in budgets]),
        P(*[t.data_ptr() for t in npoints]), P(*[t.data_ptr() for t in points_used]),
        _stream(stream))
    _check(st, "mpq_allocate_points_batched")
    return npoints, points_used


def mpq_reconstruct(codes, scales, npoints, W_hat=None, stream=None, center=None):
    """Multipoint weights (Eq. 4): W_hat [C][d] fp32, from the centres B [C] of asymmetric sets
    when given."""
    _dev(codes, "codes", torch.int8)
    k_max, C, d = codes.shape
    _dev(scales, "scales", torch.float32, (C, k_max))
    _dev(npoints, "npoints", torch.int32, (C,))
    if center is not None:
        _dev(center, "center", torch.float32, (C,))
    W_hat = W_hat if W_hat is not None else torch.empty((C, d), dtype=torch.float32,
                                                        device=codes.device)
    _dev(W_hat, "W_hat", torch.float32, (C, d))
    st = load().mpq_reconstruct(_ptr(codes), _ptr(scales), _ptr(npoints), _ptr(center), C, d,
                                k_max, _ptr(W_hat), _stream(stream))
    _check(st, "mpq_reconstruct")
    return W_hat


def mpq_center_weights(W, mode: int = MPQ_CENTER_PER_CHANNEL, center=None, Wc=None, stream=None):
    """Asymmetric sets (Eq. 1, B != 0): the centres B = the fp32 midpoint of the weights' range per
    channel or per layer, and the centred weights Wc = W - B.  Returns (center [C], Wc [C][d])."""
    _dev(W, "W", torch.float32)
    C, d = W.shape
    center = center if center is not None else torch.empty((C,), dtype=torch.float32,
                                                           device=W.device)
    Wc = Wc if Wc is not None else torch.empty((C, d), dtype=torch.float32, device=W.device)
    _dev(center, "center", torch.float32, (C,))
    _dev(Wc, "Wc", torch.float32, (C, d))
    st = load().mpq_center_weights(_ptr(W), C, d, mode, _ptr(center), _ptr(Wc), _stream(stream))
    _check(st, "mpq_center_weights")
    return center, Wc


def mpq_status_string(status: int) -> str:
    return load().mpq_status_string(status).decode()


def mpq_version() -> int:
    return load().mpq_version()


def mpq_device_status(stream=None):
    """Synchronizes the stream and takes the current device's timeout word (and, in the checked
    build, the bounds-check counts): 0 if no bounded wait of a tensor-core kernel gave up and no
    check failed since the last call, else the MPQ_TIMEOUT_* bits | MPQ_FAULT_BOUNDS."""
    flags = ctypes.c_uint(0)
    st = load().mpq_device_status(_stream(stream), ctypes.byref(flags))
    if st not in (0, 5, 7):
        _check(st, "mpq_device_status")
    return int(flags.value)


def mpq_build_options() -> int:
    """MPQ_BUILD_* bits of the loaded library (MPQ_BUILD_CHECK_BOUNDS for the checked build)."""
    return int(load().mpq_build_options())


def mpq_last_error() -> str:
    return load().mpq_last_error().decode(errors="replace")


def mpq_set_wait_limit(clocks: int):
    """Clock budget of every bounded device wait of later launches (<= 0: the default)."""
    _check(load().mpq_set_wait_limit(int(clocks)), "mpq_set_wait_limit")


def mpq_test_withhold_copies(on: bool):
    """Test hook: the output-error contraction's copy thread issues no copies while on."""
    _check(load().mpq_test_withhold_copies(1 if on else 0), "mpq_test_withhold_copies")
