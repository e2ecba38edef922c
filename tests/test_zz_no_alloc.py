"""mpq_output_error_noalloc: the output error for callers that cannot allocate device memory while
they run (a memory budget fixed up front, a framework that owns the stream-ordered pool, a pool
that is switched off).  Its range table lives in one fixed array inside the library instead of the
pool.  Checked through the C ABI against the pool-scratch entry point (bit for bit) and against
the oracle's double-precision Eq. 11 (1e-5 relative), on two calls in a row of each shape.

Collected last on purpose: every call of this entry point shares the library's fixed array, so
no other test's call may overlap it; and if it fails, a run that stops at the first failure has
already run every other test."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu

VALUE_RTOL = 1e-5


@pytest.mark.parametrize("C,d,N,K", [(130, 256, 600, 4), (64, 576, 1024, 8)])
def test_noalloc_matches_pool_scratch_and_oracle(gpu, oracle, C, d, N, K):
    W = wlm.random_weights(C, d, 5 * C + d, "normal")
    q = oracle.quantize_layer(W, 4, 32, K)
    X = wlm.random_calibration(N, d, 3 + d)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(gpu)
    args = (t(X), t(W), t(q["codes"]), t(q["scales"]), K)
    ref = binding.mpq_output_error(*args)
    first = binding.mpq_output_error_noalloc(*args)
    second = binding.mpq_output_error_noalloc(*args)
    torch.cuda.synchronize()
    assert torch.equal(first, ref) and torch.equal(second, ref)
    err_or = oracle.output_error(X, 1, W, q["codes"], q["scales"], K)
    for got in (first, second):
        g = got.cpu().numpy().astype(np.float64)
        rel = np.abs(g - err_or) / np.maximum(np.abs(err_or), 1e-300)
        assert float(rel.max()) <= VALUE_RTOL, f"max rel diff {float(rel.max()):.3e}"


def test_noalloc_rejects_oversize_table(gpu):
    C = binding.MPQ_NOALLOC_RANGE_WORDS // 3 + 1          # 1 + 3C words > the fixed array
    W = torch.zeros((C, 16), dtype=torch.float32, device=gpu)
    codes = torch.zeros((2, C, 16), dtype=torch.int8, device=gpu)
    scales = torch.zeros((C, 2), dtype=torch.float32, device=gpu)
    X = torch.zeros((8, 16), dtype=torch.float32, device=gpu)
    with pytest.raises(binding.MPQError) as e:
        binding.mpq_output_error_noalloc(X, W, codes, scales, 2)
    assert e.value.status == 3
    err = binding.mpq_output_error(X, W, codes, scales, 2)    # the pool path has no such limit
    torch.cuda.synchronize()
    assert torch.all(err == 0)
