"""Every kernel of the library on small seeded inputs, for the checked-build test
(tests/test_gpu_checked.py).

hot_path_outputs() runs each C-ABI entry point once (each kernel family and its variants: the
greedy search's lattice, event, direct and caller-grid forms, the contraction's CTA-pair,
single-CTA and per-channel forms, allocation single and batched, reconstruction, centres,
clipping, the adaptive grid, packing and integer inference on both of its paths) and returns
every output as numpy arrays, with the device status taken at the end.  corrupt_packed_channel()
plants an out-of-range channel index in a packed layer and runs inference into a padded output,
so that the skipped store is visible.

Run as a script (``MPQ_LIBRARY=<checked .so> python tests/_checked_run.py out.npz``) it saves
both results, so that a test can compare a checked-build process with the normal build.
"""
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2002_09049_gb300 import binding, workloads as wlm  # noqa: E402


def _np(t):
    return t.detach().cpu().numpy()


def hot_path_outputs(dev="cuda:0"):
    out = {}
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    W1 = wlm.random_weights(64, 576, 1, "normal")            # lattice search, CTA-pair contraction
    W2 = wlm.random_weights(16, 300, 2, "t")                 # a caller's grid
    W3 = wlm.random_weights(96, 9, 3, "laplace")             # depthwise rows: direct search
    W4 = wlm.random_weights(32, 147, 4, "normal")            # ragged d: single-CTA contraction
    rng = np.random.default_rng(11)
    W5 = (rng.integers(-60, 61, size=(4, 12)) * 2.0 ** -149).astype(np.float32)   # scale 0
    X1 = wlm.random_calibration(200, 576, 5)
    X3 = np.stack([wlm.random_calibration(50, 9, 100 + k) for k in range(96)])
    X4 = wlm.random_calibration(130, 147, 6)

    # greedy construction (Algorithm 1)
    rm1 = torch.empty((64, 5), dtype=torch.float32, device=dev)
    res1 = torch.empty((4, 64, 576), dtype=torch.float32, device=dev)
    c1, s1, r1, _ = binding.mpq_quantize_layer(t(W1), 4, 64, 4, residuals=res1, rmax=rm1)
    frac = np.sort(rng.uniform(0.05, 1.0, size=40)).astype(np.float32)
    frac[-1] = 1.0
    c2, s2, r2, _ = binding.mpq_quantize_layer(t(W2), 3, 40, 3, grid_frac=frac)
    c3, s3, r3, _ = binding.mpq_quantize_layer(t(W3), 4, 32, 4)
    c4, s4, r4, _ = binding.mpq_quantize_layer(t(W4), 4, 48, 3)
    c5, s5, r5, _ = binding.mpq_quantize_layer(t(W5), 4, 16, 2)
    for n, (c, s, r) in enumerate([(c1, s1, r1), (c2, s2, r2), (c3, s3, r3), (c4, s4, r4),
                                   (c5, s5, r5)], 1):
        out[f"codes{n}"], out[f"scales{n}"], out[f"resid_sq{n}"] = _np(c), _np(s), _np(r)
    out["residuals1"], out["rmax1"] = _np(res1), _np(rm1)

    # output error (Eq. 11): CTA pair (with and without the search's ranges), single CTA,
    # per channel, the fixed-scratch variant
    e1 = binding.mpq_output_error(t(X1), t(W1), c1, s1, 4)
    e1r = binding.mpq_output_error(t(X1), t(W1), c1, s1, 4, rmax=rm1)
    e1n = binding.mpq_output_error_noalloc(t(X1), t(W1), c1, s1, 4)
    e4 = binding.mpq_output_error(t(X4), t(W4), c4, s4, 3)
    e3 = binding.mpq_output_error(t(X3), t(W3), c3, s3, 4, groups=96)
    for k, e in dict(err1=e1, err1_rmax=e1r, err1_noalloc=e1n, err4=e4, err3=e3).items():
        out[k] = _np(e)

    # allocation (Algorithm 2): budget, threshold, batched
    n1, u1 = binding.mpq_allocate_points(e1, 4, binding.MPQ_ALLOC_BUDGET, 2.0)
    n4, u4 = binding.mpq_allocate_points(e4, 3, binding.MPQ_ALLOC_THRESHOLD, 0.5)
    nb, ub = binding.mpq_allocate_points_batched([e1, e3], 4, binding.MPQ_ALLOC_BUDGET, [1.5, 2.5])
    out.update(npoints1=_np(n1), used1=_np(u1), npoints4=_np(n4), used4=_np(u4))
    for i, (n, u) in enumerate(zip(nb, ub)):
        out[f"npoints_batch{i}"], out[f"used_batch{i}"] = _np(n), _np(u)

    # multipoint weights (Eq. 4), centres (Eq. 1)
    out["W_hat1"] = _np(binding.mpq_reconstruct(c1, s1, n1))
    out["W_hat4"] = _np(binding.mpq_reconstruct(c4, s4, n4))
    B1, Wc1 = binding.mpq_center_weights(t(W1), binding.MPQ_CENTER_PER_CHANNEL)
    B4, Wc4 = binding.mpq_center_weights(t(W4), binding.MPQ_CENTER_PER_LAYER)
    out.update(center1=_np(B1), Wc1=_np(Wc1), center4=_np(B4), Wc4=_np(Wc4))
    out["W_hat4_centered"] = _np(binding.mpq_reconstruct(c4, s4, n4, center=B4))

    # clipping factor search (Eq. 12)
    for key, (X, W, mode) in dict(clip1=(X1, W1, binding.MPQ_CLIP_PER_CHANNEL),
                                  clip4=(X4, W4, binding.MPQ_CLIP_PER_LAYER)).items():
        clip, err, best = binding.mpq_clip_search(t(X), t(W), 4, n_cand=10, mode=mode)
        out[key], out[key + "_err"], out[key + "_best"] = _np(clip), _np(err), _np(best)

    # adaptive grid (Def. 1, Eq. 10)
    ca, sa, ra, na = binding.mpq_quantize_layer_adaptive(t(W1[:6, :64]), 4, 3)
    out.update(codes_ad=_np(ca), scales_ad=_np(sa), resid_sq_ad=_np(ra), ncand_ad=_np(na))

    # packing and integer inference (Eq. 13): tensor-core path (d % 16 == 0), plain path (d = 147)
    for key, (c, s, n, d, T) in dict(y1=(c1, s1, n1, 576, 300), y4=(c4, s4, n4, 147, 70)).items():
        k_max = c.shape[0]
        lay = binding.mpq_pack_layout(_np(n), d, k_max, 4, 12)
        packed = binding.mpq_pack_points(c, s, _np(n), lay)
        Xq = t(rng.integers(-127, 128, size=(T, d)).astype(np.int8))
        out[key] = _np(binding.mpq_multipoint_linear(Xq, lay, packed))

    torch.cuda.synchronize()
    out["flags"] = np.array([binding.mpq_device_status()], dtype=np.int64)
    return out


def corrupt_packed_channel(dev="cuda:0"):
    """Inference on a packed layer whose first row names channel C + 3: the store to that
    channel's outputs must be skipped.  Y is the head of a larger buffer filled with a sentinel,
    so that a store past the layer's C rows would land in the buffer's own tail.  Returns
    (status flags, last error message, tail untouched)."""
    C, d, T, K = 64, 576, 256, 3
    W = wlm.random_weights(C, d, 21, "normal")
    c, s, _, _ = binding.mpq_quantize_layer(torch.from_numpy(W).to(dev), 4, 32, K)
    n = np.full(C, K, dtype=np.int32)
    lay = binding.mpq_pack_layout(n, d, K, 4, 12)
    packed = binding.mpq_pack_points(c, s, n, lay)
    chan = packed[lay.off_chan:lay.off_chan + 4 * lay.rows].view(torch.int32)
    chan[0] = C + 3
    X = torch.from_numpy(np.random.default_rng(22).integers(-127, 128, size=(T, d))
                         .astype(np.int8)).to(dev)
    sentinel = -123456789
    Ybuf = torch.full(((C + 8) * T,), sentinel, dtype=torch.int32, device=dev)
    Y = Ybuf[:C * T].view(C, T)
    binding.mpq_multipoint_linear(X, lay, packed, Y=Y)
    torch.cuda.synchronize()
    flags = binding.mpq_device_status()
    msg = binding.mpq_last_error()
    tail_ok = bool(torch.all(Ybuf[C * T:] == sentinel).item())
    return flags, msg, tail_ok


if __name__ == "__main__":
    res = hot_path_outputs()
    flags, msg, tail_ok = corrupt_packed_channel()
    res["corrupt_flags"] = np.array([flags], dtype=np.int64)
    res["corrupt_tail_ok"] = np.array([tail_ok])
    res["corrupt_msg"] = np.array([msg])
    res["build_options"] = np.array([binding.mpq_build_options()], dtype=np.int64)
    np.savez(sys.argv[1], **res)
