"""End-to-end parity of the whole path on the single conv-shaped layer workload and sampled
parity at full size on the ResNet-18-shaped and large-linear workloads."""
import numpy as np
import pytest
import torch

from paper_2002_09049_gb300 import binding, pipeline, workloads as wlm
from _parity import compare_err, compare_quantize

pytestmark = pytest.mark.gpu


def test_config1_end_to_end(gpu, oracle):
    wl = wlm.WORKLOADS["c1"]
    W = wlm.make_weights(wl, 0)
    X = wlm.make_calibration(wl, 0)
    spec = pipeline.LayerSpec(C=64, d=576, N=512, bits=4, G=wl.G, k_max=wl.k_max,
                              budget_or_eps=wl.beta)
    plan = pipeline.LayerPlan(spec, gpu)
    Wd, Xd = torch.from_numpy(W).to(gpu), torch.from_numpy(X).to(gpu)
    plan.run_device(Wd, Xd)
    torch.cuda.synchronize()
    gpu_q = dict(codes=plan.codes.cpu().numpy(), scales=plan.scales.cpu().numpy(),
                 resid_sq=plan.resid_sq.cpu().numpy())
    orc = oracle.quantize_layer(W, 4, wl.G, wl.k_max)
    rep = compare_quantize(W, gpu_q, orc, 4, wl.G, wl.k_max, oracle=oracle)
    err_or = oracle.output_error(X, 1, W, orc["codes"], orc["scales"], wl.k_max)
    err_gpu = plan.err.cpu().numpy()
    if rep["near_ties"] == 0:
        compare_err(err_gpu, err_or)
        # allocation on the GPU's own error table must equal the sequential loop on that table
        n_or, used_or = oracle.allocate_budget(err_gpu, wl.k_max, wl.beta)
        assert np.array_equal(plan.npoints.cpu().numpy(), n_or)
        assert int(plan.points_used.item()) == used_or == int(np.floor(wl.beta * 64 + 0.5))
        What = oracle.reconstruct(orc["codes"], orc["scales"], n_or)
        assert np.array_equal(plan.W_hat.cpu().numpy(), What)


def test_run_host_matches_device(gpu):
    wl = wlm.WORKLOADS["c1"]
    W = torch.from_numpy(wlm.make_weights(wl, 0)).pin_memory()
    X = torch.from_numpy(wlm.make_calibration(wl, 0)).pin_memory()
    spec = pipeline.LayerSpec(C=64, d=576, N=512, G=wl.G, k_max=wl.k_max, budget_or_eps=wl.beta)
    plan = pipeline.LayerPlan(spec, gpu)
    Wd, Xd = torch.empty_like(W, device=gpu), torch.empty_like(X, device=gpu)
    h = plan.run_host(W, X, Wd, Xd)
    torch.cuda.synchronize()
    assert torch.equal(h["codes"], plan.codes.cpu()) and torch.equal(h["npoints"],
                                                                     plan.npoints.cpu())


def sample_channels(C, rng, edge=16, frac=0.02):
    idx = set(range(min(edge, C))) | set(range(max(0, C - edge), C))
    idx |= set(rng.choice(C, size=max(1, int(frac * C)), replace=False).tolist())
    return sorted(idx)


@pytest.mark.parametrize("key,layers", [("c2", [0, 9, 16, 20]), ("c5", [1]), ("c4", [0, 1, 49, 52]),
                                        ("c3", [3, 40])])
def test_full_size_sampled(gpu, oracle, key, layers):
    """Full-size layers on the GPU in the bench's launch configuration; the oracle checks a
    sample of channels (first/last 16 and 2 % at random) of codes, scales and output errors."""
    wl = wlm.WORKLOADS[key]
    rng = np.random.default_rng(0)
    for li in layers:
        layer = wl.layers[li]
        W = wlm.make_weights(wl, li)
        X = wlm.make_calibration(wl, li)
        bits = wl.bits[-1]
        spec = pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, groups=layer.groups,
                                  bits=bits, G=wl.G, k_max=wl.k_max, budget_or_eps=wl.beta)
        plan = pipeline.LayerPlan(spec, gpu)
        plan.run_device(torch.from_numpy(W).to(gpu), torch.from_numpy(X).to(gpu))
        torch.cuda.synchronize()
        ch = sample_channels(layer.C, rng)
        gq = dict(codes=plan.codes.cpu().numpy(), scales=plan.scales.cpu().numpy(),
                  resid_sq=plan.resid_sq.cpu().numpy())
        orc = {}
        sub = W[ch]
        o = oracle.quantize_layer(sub, bits, wl.G, wl.k_max, threads=8)
        gsub = dict(codes=gq["codes"][:, ch], scales=gq["scales"][ch], resid_sq=gq["resid_sq"][ch])
        rep = compare_quantize(sub, gsub, o, bits, wl.G, wl.k_max, oracle=oracle)
        # output error of the sampled channels from the GPU's codes (same inputs on both sides)
        Xs = X[ch] if layer.groups > 1 else X
        e_or = oracle.output_error(Xs, len(ch) if layer.groups > 1 else 1, sub, gsub["codes"],
                                   gsub["scales"], wl.k_max, threads=8)
        compare_err(plan.err.cpu().numpy()[ch], e_or)
        # allocation on the GPU's error table is exactly the sequential loop
        n_or, used_or = oracle.allocate_budget(plan.err.cpu().numpy(), wl.k_max, wl.beta)
        assert np.array_equal(plan.npoints.cpu().numpy(), n_or)
        assert int(plan.points_used.item()) == used_or


def test_network_plan_streams_match_single_stream(gpu):
    """Layers spread over 8 streams give bit-identical outputs to one stream (layers are
    independent; every kernel is deterministic)."""
    wl = wlm.WORKLOADS["c2"]
    idx = [0, 1, 5, 7, 12, 16, 20]
    specs, Ws, Xs = [], [], []
    for li in idx:
        layer = wl.layers[li]
        specs.append(pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, bits=4, G=wl.G,
                                        k_max=wl.k_max, budget_or_eps=wl.beta))
        Ws.append(torch.from_numpy(wlm.make_weights(wl, li)).to(gpu))
        Xs.append(torch.from_numpy(wlm.make_calibration(wl, li)).to(gpu))
    many = pipeline.NetworkPlan(specs, gpu, n_streams=8).run_device(Ws, Xs)
    one = pipeline.NetworkPlan(specs, gpu, n_streams=1).run_device(Ws, Xs)
    # every layer's allocation per layer instead of in one batched launch
    per_layer = pipeline.NetworkPlan(specs, gpu, n_streams=8, batch_alloc=False).run_device(Ws, Xs)
    torch.cuda.synchronize()
    assert many.batch_alloc and not per_layer.batch_alloc
    for a, b, c in zip(many.plans, one.plans, per_layer.plans):
        for name in ("codes", "scales", "resid_sq", "err", "npoints", "points_used", "W_hat"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name
            assert torch.equal(getattr(a, name), getattr(c, name)), name


def test_captured_graph_matches_launches(gpu):
    """A CUDA-graph replay of the multi-stream step gives bit-identical outputs to launching it."""
    wl = wlm.WORKLOADS["c2"]
    idx = [0, 5, 16, 20]
    specs, Ws, Xs = [], [], []
    for li in idx:
        layer = wl.layers[li]
        specs.append(pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, bits=4, G=wl.G,
                                        k_max=wl.k_max, budget_or_eps=wl.beta))
        Ws.append(torch.from_numpy(wlm.make_weights(wl, li)).to(gpu))
        Xs.append(torch.from_numpy(wlm.make_calibration(wl, li)).to(gpu))
    ref = pipeline.NetworkPlan(specs, gpu, n_streams=4).run_device(Ws, Xs)
    torch.cuda.synchronize()
    ref_out = [{n: getattr(p, n).clone() for n in ("codes", "scales", "err", "npoints", "W_hat")}
               for p in ref.plans]
    net = pipeline.NetworkPlan(specs, gpu, n_streams=4)
    cap = pipeline.CapturedNetwork(net, Ws, Xs)
    for p in net.plans:                 # poison the outputs: the replay must rewrite them all
        for n in ("codes", "scales", "err", "npoints", "W_hat"):
            getattr(p, n).fill_(0)
    cap.replay()
    torch.cuda.synchronize()
    for p, r in zip(net.plans, ref_out):
        for n, v in r.items():
            assert torch.equal(getattr(p, n), v), n


@pytest.mark.parametrize("center", [-1, 0])
def test_network_run_host_matches_device(gpu, center):
    """The end-to-end network call (inputs copied in on one stream, outputs copied out on another,
    kernels on the compute streams in between) returns exactly what the device-resident call
    computes, on every repetition."""
    wl = wlm.WORKLOADS["c2"]
    idx = [0, 3, 9, 16, 20]
    specs, Whs, Xhs = [], [], []
    for li in idx:
        layer = wl.layers[li]
        specs.append(pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, bits=4, G=wl.G,
                                        k_max=wl.k_max, budget_or_eps=wl.beta, center=center))
        Whs.append(torch.from_numpy(wlm.make_weights(wl, li)).pin_memory())
        Xhs.append(torch.from_numpy(wlm.make_calibration(wl, li)).pin_memory())
    ref = pipeline.NetworkPlan(specs, gpu, n_streams=3).run_device(
        [w.to(gpu) for w in Whs], [x.to(gpu) for x in Xhs])
    torch.cuda.synchronize()
    net = pipeline.NetworkPlan(specs, gpu, n_streams=3)
    Wds = [torch.empty_like(w, device=gpu) for w in Whs]
    Xds = [torch.empty_like(x, device=gpu) for x in Xhs]
    for _ in range(2):
        outs = net.run_host(Whs, Xhs, Wds, Xds)
        torch.cuda.synchronize()
        for h, p in zip(outs, ref.plans):
            assert torch.equal(h["codes"], p.codes.cpu()) and torch.equal(h["scales"], p.scales.cpu())
            assert torch.equal(h["npoints"], p.npoints.cpu())
            assert int(h["points_used"].item()) == int(p.points_used.item())
            if center >= 0:
                assert torch.equal(h["center"], p.center.cpu())


def test_captured_end_to_end_matches_device(gpu):
    """The captured end-to-end step (copies in, path, copies out) writes the same host outputs as
    the device-resident call, and a replay after new host inputs picks them up."""
    wl = wlm.WORKLOADS["c2"]
    idx = [1, 9, 16]
    specs, Whs, Xhs = [], [], []
    for li in idx:
        layer = wl.layers[li]
        specs.append(pipeline.LayerSpec(C=layer.C, d=layer.d, N=wl.n_calib, bits=4, G=wl.G,
                                        k_max=wl.k_max, budget_or_eps=wl.beta))
        Whs.append(torch.from_numpy(wlm.make_weights(wl, li)).pin_memory())
        Xhs.append(torch.from_numpy(wlm.make_calibration(wl, li)).pin_memory())
    net = pipeline.NetworkPlan(specs, gpu, n_streams=2)
    Wds = [torch.empty_like(w, device=gpu) for w in Whs]
    Xds = [torch.empty_like(x, device=gpu) for x in Xhs]
    cap = pipeline.CapturedNetwork(net, Wds, Xds, host=(Whs, Xhs))
    for scale in (1.0, 0.5):
        for w in Whs:
            w.mul_(scale)
        cap.replay()
        torch.cuda.synchronize()
        ref = pipeline.NetworkPlan(specs, gpu, n_streams=1).run_device(
            [w.to(gpu) for w in Whs], [x.to(gpu) for x in Xhs])
        torch.cuda.synchronize()
        for h, p in zip(cap.host_outputs(), ref.plans):
            assert torch.equal(h["codes"], p.codes.cpu()) and torch.equal(h["scales"], p.scales.cpu())
            assert torch.equal(h["npoints"], p.npoints.cpu())
