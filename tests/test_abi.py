"""The C-ABI library builds, loads without a GPU, exports every symbol include/*.h declares, and
rejects invalid arguments on the host before touching the device (no GPU needed)."""
import ctypes
import glob
import os
import re

import pytest

from paper_2002_09049_gb300 import _build, binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^[A-Za-z_][\w \t\*]*?\b(mpq_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return binding.load()


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("mpq_quantize_layer", "mpq_output_error", "mpq_allocate_points", "mpq_reconstruct",
              "mpq_clip_search", "mpq_center_weights", "mpq_pack_layout", "mpq_pack_points",
              "mpq_multipoint_linear"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    raw = ctypes.CDLL(_build.LIB)
    for name in declared_functions():
        assert hasattr(raw, name), name
        assert name in binding.SIGNATURES, name


def test_status_strings(lib):
    assert lib.mpq_status_string(0) == b"MPQ_OK"
    assert lib.mpq_status_string(3) == b"MPQ_ERR_UNSUPPORTED"
    assert lib.mpq_status_string(7) == b"MPQ_ERR_BOUNDS"
    assert lib.mpq_version() >= 100


def test_checked_build_exports_and_reports_its_option(lib):
    """The checked build (-DMPQ_CHECK_BOUNDS) compiles, loads without a GPU, exports every
    declared symbol and says what it is through mpq_build_options; the normal build says 0."""
    raw = ctypes.CDLL(_build.build(checked=True))
    for name in declared_functions():
        assert hasattr(raw, name), name
    raw.mpq_build_options.restype = ctypes.c_uint
    assert raw.mpq_build_options() == binding.MPQ_BUILD_CHECK_BOUNDS
    assert binding.mpq_build_options() == 0


P = ctypes.c_void_p
FAKE = P(0x1000)  # never dereferenced: every call below fails validation on the host first


@pytest.mark.parametrize("kwargs,status", [
    (dict(bits=1), 1), (dict(bits=9), 3), (dict(G=0), 1), (dict(G=1025), 3), (dict(k_max=0), 1),
    (dict(k_max=17), 3), (dict(d=0), 1), (dict(d=8193), 3), (dict(C=-1), 1),
    (dict(W=None), 1), (dict(codes=None), 1), (dict(scales=None), 1),
])
def test_quantize_validation(lib, kwargs, status):
    a = dict(W=FAKE, C=4, d=16, bits=4, G=8, grid=None, k_max=2, codes=FAKE, scales=FAKE)
    a.update(kwargs)
    st = lib.mpq_quantize_layer(a["W"], a["C"], a["d"], a["bits"], a["G"], a["grid"], a["k_max"],
                                a["codes"], a["scales"], None, None, None, None)
    assert st == status
    assert lib.mpq_last_error() != b""


@pytest.mark.parametrize("grid", [[0.5, 0.25, 1.0], [0.0, 0.5, 1.0], [0.5, 0.5, 1.0],
                                  [0.5, 0.75, 1.5], [0.5, float("nan"), 1.0]])
def test_quantize_rejects_bad_grid(lib, grid):
    g = (ctypes.c_float * 3)(*grid)
    st = lib.mpq_quantize_layer(FAKE, 4, 16, 4, 3, g, 2, FAKE, FAKE, None, None, None, None)
    assert st == 1


def test_empty_layer_is_a_no_op(lib):
    assert lib.mpq_quantize_layer(None, 0, 16, 4, 8, None, 2, None, None, None, None, None,
                                  None) == 0
    assert lib.mpq_output_error(None, 5, 1, None, None, None, None, 0, 16, 2, None, None) == 0
    assert lib.mpq_reconstruct(None, None, None, None, 0, 16, 2, None, None) == 0
    assert lib.mpq_center_weights(None, 0, 16, 0, None, None, None) == 0


@pytest.mark.parametrize("args,status", [
    ((FAKE, 0, 1, FAKE, FAKE, FAKE, 4, 16, 2, FAKE), 1),    # N = 0
    ((FAKE, 8, 3, FAKE, FAKE, FAKE, 4, 16, 2, FAKE), 1),    # groups not in {1, C}
    ((None, 8, 1, FAKE, FAKE, FAKE, 4, 16, 2, FAKE), 1),    # X NULL
    ((FAKE, 8, 1, FAKE, FAKE, FAKE, 4, 16, 2, None), 1),    # err NULL
])
def test_output_error_validation(lib, args, status):
    assert lib.mpq_output_error(*args[:6], None, *args[6:], None) == status


def test_output_error_noalloc_validation(lib):
    """The fixed-scratch entry point validates like mpq_output_error and rejects, on the host, a
    range table larger than its buffer (16-byte aligned fake pointers and d % 16 == 0 select the
    tensor-core path, whose table has 1 + C (k_max+1) words)."""
    f = lib.mpq_output_error_noalloc
    assert f(FAKE, 0, 1, FAKE, FAKE, FAKE, 4, 16, 2, FAKE, None) == 1                  # N = 0
    assert f(None, 8, 1, FAKE, FAKE, FAKE, 4, 16, 2, FAKE, None) == 1                  # X NULL
    assert f(FAKE, 8, 1, FAKE, FAKE, FAKE, 0, 16, 2, FAKE, None) == 0                  # C = 0
    C = binding.MPQ_NOALLOC_RANGE_WORDS // 3 + 1                                       # 3C + 1 > words
    assert f(FAKE, 8, 1, FAKE, FAKE, FAKE, C, 16, 2, FAKE, None) == 3


@pytest.mark.parametrize("d,bits,eta,cap,status", [
    (8193, 4, 2.0 ** -10, 100, 3),        # longer than MPQ_MAX_DIM
    (1024, 8, 2.0 ** -10, 100, 3),        # d * Qmax above MPQ_ADAPTIVE_MAX_THRESHOLDS
    (9, 9, 2.0 ** -10, 100, 3),           # bits above the limit
    (9, 1, 2.0 ** -10, 100, 1),
    (9, 4, 0.0, 100, 1),                  # eta must be > 0
    (9, 4, float("nan"), 100, 2),
    (9, 4, 2.0 ** -10, 0, 1),             # max_cand >= 1
])
def test_quantize_adaptive_validation(lib, d, bits, eta, cap, status):
    assert lib.mpq_quantize_layer_adaptive(FAKE, 4, d, bits, 3, eta, cap, FAKE, FAKE, None, None,
                                           None) == status


@pytest.mark.parametrize("mode,val,status", [
    (2, 1.0, 1), (0, float("nan"), 2), (0, float("inf"), 2), (0, -0.5, 1), (1, float("nan"), 2),
])
def test_allocate_validation(lib, mode, val, status):
    assert lib.mpq_allocate_points(FAKE, 4, 3, mode, val, FAKE, None, None) == status


def test_allocate_requires_outputs(lib):
    assert lib.mpq_allocate_points(FAKE, 4, 3, 0, 1.5, None, None, None) == 1


def test_reconstruct_validation(lib):
    assert lib.mpq_reconstruct(FAKE, FAKE, None, None, 4, 16, 2, FAKE, None) == 1
    assert lib.mpq_reconstruct(FAKE, FAKE, FAKE, FAKE, 4, 16, 0, FAKE, None) == 1


@pytest.mark.parametrize("kwargs,status", [
    (dict(mode=2), 1), (dict(mode=-1), 1), (dict(d=0), 1), (dict(C=-1), 1), (dict(W=None), 1),
    (dict(center=None), 1), (dict(Wc=None), 1),
])
def test_center_validation(lib, kwargs, status):
    a = dict(W=FAKE, C=4, d=16, mode=1, center=FAKE, Wc=FAKE)
    a.update(kwargs)
    assert lib.mpq_center_weights(a["W"], a["C"], a["d"], a["mode"], a["center"], a["Wc"],
                                  None) == status
    assert lib.mpq_last_error() != b""


@pytest.mark.parametrize("kwargs,status", [
    (dict(N=0), 1), (dict(groups=3), 1), (dict(bits=1), 1), (dict(bits=9), 3), (dict(n_cand=0), 1),
    (dict(n_cand=33), 3), (dict(mode=2), 1), (dict(d=0), 1), (dict(d=8193), 3), (dict(X=None), 1),
    (dict(clip=None), 1), (dict(err=None), 1), (dict(best=None), 1),
])
def test_clip_search_validation(lib, kwargs, status):
    a = dict(X=FAKE, N=8, groups=1, W=FAKE, C=4, d=16, bits=4, n_cand=20, mode=0, clip=FAKE,
             err=FAKE, best=FAKE)
    a.update(kwargs)
    st = lib.mpq_clip_search(a["X"], a["N"], a["groups"], a["W"], a["C"], a["d"], a["bits"],
                             a["n_cand"], a["mode"], a["clip"], a["err"], a["best"], None)
    assert st == status
    assert lib.mpq_last_error() != b""


def test_clip_search_empty_layer(lib):
    assert lib.mpq_clip_search(None, 8, 1, None, 0, 16, 4, 20, 1, None, None, None, None) == 0


def test_pack_layout_groups_channels(lib):
    """Host-only layout: channels grouped by the power of two >= n_k (n_k = 0 takes one row), 128/R
    channels per 128-row tile, rows padded to 64 elements, byte offsets in order."""
    assert ctypes.sizeof(binding.PackedLayout) == 10 * 4 + 7 * 8   # 9 ints + padding, 7 size_t
    npts = [1] * 200 + [2] * 70 + [3] * 5 + [0] * 3 + [16]
    lay = binding.mpq_pack_layout(npts, 100, 16, 4, 12)
    tiles = -(-203 // 128) + -(-70 // 64) + -(-5 // 32) + 1   # R = 1, 2, 4, 16
    assert (lay.C, lay.d, lay.d_pad, lay.tiles, lay.rows) == (279, 100, 128, tiles, 128 * tiles)
    assert lay.centered == 0
    assert lay.off_coef < lay.off_chan < lay.off_point < lay.off_tile <= lay.off_center
    assert lay.off_center < lay.off_codes < lay.bytes
    assert lay.off_codes % 1024 == 0
    assert lay.bytes == lay.off_codes + lay.rows * lay.d_pad * 2
    cen = binding.mpq_pack_layout(npts, 100, 16, 4, 12, centered=True)
    assert cen.centered == 1 and cen.off_center == lay.off_center
    assert cen.off_codes >= cen.off_center + 279 * 4 and cen.off_codes % 1024 == 0


@pytest.mark.parametrize("kwargs,status", [
    (dict(p=31), 1), (dict(p=-1), 1), (dict(bits=1), 1), (dict(bits=9), 3), (dict(k_max=17), 3),
    (dict(d=0), 1), (dict(npoints=None), 1), (dict(layout=None), 1), (dict(centered=2), 1),
])
def test_pack_layout_validation(lib, kwargs, status):
    n = (ctypes.c_int * 3)(1, 2, 3)
    lay = binding.PackedLayout()
    a = dict(npoints=n, C=3, d=32, k_max=4, bits=4, p=12, centered=0, layout=ctypes.byref(lay))
    a.update(kwargs)
    assert lib.mpq_pack_layout(a["npoints"], a["C"], a["d"], a["k_max"], a["bits"], a["p"],
                               a["centered"], a["layout"]) == status


def test_pack_and_linear_validation(lib):
    lay = binding.mpq_pack_layout([1, 2], 32, 4, 4, 12)
    assert lib.mpq_pack_points(None, FAKE, None, FAKE, ctypes.byref(lay), FAKE, None) == 1
    assert lib.mpq_pack_points(FAKE, FAKE, None, FAKE, None, FAKE, None) == 1
    assert lib.mpq_pack_points(FAKE, FAKE, FAKE, FAKE, ctypes.byref(lay), FAKE, None) == 1  # not centred
    cen = binding.mpq_pack_layout([1, 2], 32, 4, 4, 12, centered=True)
    assert lib.mpq_pack_points(FAKE, FAKE, None, FAKE, ctypes.byref(cen), FAKE, None) == 1
    assert lib.mpq_multipoint_linear(FAKE, 0, ctypes.byref(lay), FAKE, FAKE, None) == 1
    assert lib.mpq_multipoint_linear(None, 4, ctypes.byref(lay), FAKE, FAKE, None) == 1
    assert lib.mpq_multipoint_linear(FAKE, 4, None, FAKE, FAKE, None) == 1


def test_batched_allocation_validation(lib):
    f = lib.mpq_allocate_points_batched
    errs = (ctypes.c_void_p * 2)(0x1000, 0x2000)
    Cs = (ctypes.c_int * 2)(4, 8)
    vals = (ctypes.c_double * 2)(1.5, 1.5)
    npts = (ctypes.c_void_p * 2)(0x3000, 0x4000)
    assert f(0, None, None, 4, 0, None, None, None, None) == 0                      # nothing
    assert f(65, errs, Cs, 4, 0, vals, npts, None, None) == 3                      # > MPQ_MAX_BATCH
    assert f(2, None, Cs, 4, 0, vals, npts, None, None) == 1                       # err array NULL
    assert f(2, errs, Cs, 4, 2, vals, npts, None, None) == 1                       # bad mode
    assert f(2, errs, Cs, 0, 0, vals, npts, None, None) == 1                       # k_max = 0
    bad = (ctypes.c_double * 2)(1.5, float("nan"))
    assert f(2, errs, Cs, 4, 0, bad, npts, None, None) == 2                        # NaN budget
    neg = (ctypes.c_double * 2)(-1.0, 1.5)
    assert f(2, errs, Cs, 4, 0, neg, npts, None, None) == 1                        # budget < 0
    nulls = (ctypes.c_void_p * 2)(0x3000, None)
    assert f(2, errs, Cs, 4, 0, vals, nulls, None, None) == 1                      # npoints[1] NULL
