"""mpq_output_error_noalloc (the output error with its range table in one fixed device buffer
inside the library, no allocation) against mpq_output_error (stream-ordered scratch): two calls of
different shapes, one after the other on the same stream, give bit-identical results.  Collected
last on purpose: it shares the library's fixed buffer, so no other test's call overlaps it."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, workloads as wlm

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("C,d,N,K", [(130, 256, 600, 4), (64, 576, 1024, 8)])
def test_noalloc_matches_pool_scratch(gpu, oracle, C, d, N, K):
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


def test_noalloc_rejects_oversize_table(gpu):
    C = binding.MPQ_NOALLOC_RANGE_WORDS // 3 + 1          # 1 + 3C words > the fixed buffer
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
