"""The checked build (-DMPQ_CHECK_BOUNDS, libmpq_checked.so; include/mpq.h): every kernel checks
the indices it computes -- global stores against their outputs' extents, data-dependent
shared-memory indices against their arrays, the carve-up of dynamic shared memory against the
launch's share, tile-copy coordinates against the 16-byte rule -- and counts and skips a failed
access instead of trapping.

A child process loads the checked library (MPQ_LIBRARY) and runs every entry point on small
seeded inputs (tests/_checked_run.py).  Checked here: the library is the checked build; no check
failed on any kernel; every output equals the normal build's, bit for bit, except the greedy
search's ||r||^2, an fp32 tree sum whose shape follows the warps per channel (a launch choice
made from the kernel's occupancy, which the checks' registers can change), held to that tree's
2^-18 relative bound; and a packed layer with an out-of-range channel index has its store
skipped and reported as MPQ_FAULT_BOUNDS, naming the inference kernel's source, with nothing
written past the output (the output is the head of a larger buffer, so that even a store that
escaped the check would stay inside memory the test owns)."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2002_09049_gb300 import _build, binding

import _checked_run

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
RESID_RTOL = 2.0 ** -18


@pytest.fixture(scope="module")
def checked(gpu, tmp_path_factory):
    lib = _build.build(checked=True)
    out = tmp_path_factory.mktemp("checked") / "checked.npz"
    env = dict(os.environ, MPQ_LIBRARY=lib)
    r = subprocess.run([sys.executable, os.path.join(HERE, "_checked_run.py"), str(out)], env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-4000:]
    with np.load(out) as z:
        return {k: z[k] for k in z.files}


def test_child_ran_the_checked_build(checked):
    assert int(checked["build_options"][0]) & binding.MPQ_BUILD_CHECK_BOUNDS
    assert binding.mpq_build_options() == 0          # this process: the normal build


def test_no_kernel_fails_a_check(checked):
    assert int(checked["flags"][0]) == 0


def test_checked_outputs_equal_the_normal_build(gpu, checked):
    normal = _checked_run.hot_path_outputs()
    assert int(normal["flags"][0]) == 0
    assert set(normal) <= set(checked)
    for key, ref in normal.items():
        got = checked[key]
        assert got.shape == ref.shape and got.dtype == ref.dtype, key
        if key.startswith("resid_sq"):
            np.testing.assert_allclose(got, ref, rtol=RESID_RTOL, atol=0, err_msg=key)
        else:
            assert np.array_equal(got, ref, equal_nan=ref.dtype.kind == "f"), key


def test_out_of_range_channel_is_skipped_and_reported(checked):
    flags = int(checked["corrupt_flags"][0])
    assert flags == binding.MPQ_FAULT_BOUNDS
    assert "multipoint.cu" in str(checked["corrupt_msg"][0])
    assert bool(checked["corrupt_tail_ok"][0])
