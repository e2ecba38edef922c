"""One layer through the whole hot path: greedy points (Algorithm 1), output error (Eq. 11),
point allocation (Algorithm 2), multipoint weights (Eq. 4); with asymmetric sets (Eq. 1, B != 0)
the weights are centred first and the points approximate the centred weights.

``LayerPlan`` owns the device output buffers of one layer so that repeated runs allocate nothing;
``run_device`` enqueues the four C-ABI calls on one stream; ``run_host`` is the end-to-end call
for host data: copies W and X in from (pinned) host memory, runs the path and copies the durable
result (codes, scales, point counts) back out.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import binding


@dataclass
class LayerSpec:
    C: int
    d: int
    N: int
    groups: int = 1
    bits: int = 4
    G: int = 64
    k_max: int = 4
    mode: int = binding.MPQ_ALLOC_BUDGET
    budget_or_eps: float = 1.5
    center: int = -1        # -1 symmetric sets, else MPQ_CENTER_PER_CHANNEL / _PER_LAYER


class LayerPlan:
    def __init__(self, spec: LayerSpec, device, with_reconstruct: bool = True, counts=None):
        """counts, if given: (npoints [C], points_used [1]) int32 device views to write the
        point counts into (a network plan keeps every layer's counts in one buffer)."""
        self.spec = spec
        s = spec
        dev = torch.device(device)
        self.codes = torch.empty((s.k_max, s.C, s.d), dtype=torch.int8, device=dev)
        self.scales = torch.empty((s.C, s.k_max), dtype=torch.float32, device=dev)
        self.resid_sq = torch.empty((s.C, s.k_max + 1), dtype=torch.float32, device=dev)
        # max |r| of every residual vector: the output error's operand ranges, kept from the
        # greedy search so that they are not measured again
        self.rmax = torch.empty((s.C, s.k_max + 1), dtype=torch.float32, device=dev)
        self.err = torch.empty((s.C, s.k_max + 1), dtype=torch.float32, device=dev)
        if counts is None:
            self.npoints = torch.empty((s.C,), dtype=torch.int32, device=dev)
            self.points_used = torch.empty((1,), dtype=torch.int32, device=dev)
        else:
            self.npoints, self.points_used = counts
        self.W_hat = torch.empty((s.C, s.d), dtype=torch.float32, device=dev) \
            if with_reconstruct else None
        self.center = self.Wc = None
        if s.center >= 0:
            self.center = torch.empty((s.C,), dtype=torch.float32, device=dev)
            self.Wc = torch.empty((s.C, s.d), dtype=torch.float32, device=dev)
        self._host = None

    # -- device-resident inputs ---------------------------------------------------------------
    def run_device(self, W, X, stream=None, grid_frac=None, timing=None, x_ready=None,
                   finish=True):
        """Enqueue the four calls (five with centring) on ``stream``.  timing(phase), if given, is
        called before the first call (phase 0) and after the centring (1, also when there is
        none), the greedy points (2), the output error (3), the allocation (4) and the
        reconstruction (5), e.g. to record CUDA events.  x_ready, if given, is a CUDA event the
        stream waits on before the output error, the first call that reads X (its copy may still
        be in flight while the greedy search runs).  finish=False stops after the output error
        (a network plan then allocates every layer's points in one call, and reconstructs)."""
        s = self.spec
        tick = timing or (lambda ph: None)
        tick(0)
        if self.center is not None:
            binding.mpq_center_weights(W, s.center, center=self.center, Wc=self.Wc, stream=stream)
            W = self.Wc
        tick(1)
        binding.mpq_quantize_layer(W, s.bits, s.G, s.k_max, grid_frac=grid_frac, codes=self.codes,
                                   scales=self.scales, resid_sq=self.resid_sq, rmax=self.rmax,
                                   stream=stream)
        tick(2)
        if x_ready is not None:
            (stream or torch.cuda.current_stream()).wait_event(x_ready)
        binding.mpq_output_error(X, W, self.codes, self.scales, s.k_max, groups=s.groups,
                                 err=self.err, stream=stream, rmax=self.rmax)
        tick(3)
        if not finish:
            return self
        binding.mpq_allocate_points(self.err, s.k_max, s.mode, s.budget_or_eps,
                                    npoints=self.npoints, points_used=self.points_used,
                                    stream=stream)
        tick(4)
        self.run_reconstruct(stream)
        tick(5)
        return self

    def run_reconstruct(self, stream=None):
        """The multipoint weights (Eq. 4) from the allocated point counts, if kept."""
        if self.W_hat is not None:
            binding.mpq_reconstruct(self.codes, self.scales, self.npoints, W_hat=self.W_hat,
                                    stream=stream, center=self.center)
        return self

    # -- host inputs / outputs (end to end) ----------------------------------------------------
    def host_buffers(self, pin: bool = True, counts=None):
        """Pinned host buffers for the durable result of one run (counts: host views for the
        point counts, as in __init__)."""
        if self._host is None:
            s = self.spec
            mk = lambda shape, dt: torch.empty(shape, dtype=dt, pin_memory=pin)
            npts, used = counts if counts is not None else (mk((s.C,), torch.int32),
                                                            mk((1,), torch.int32))
            self._host = dict(codes=mk((s.k_max, s.C, s.d), torch.int8),
                              scales=mk((s.C, s.k_max), torch.float32),
                              npoints=npts, points_used=used)
            if self.center is not None:
                self._host["center"] = mk((s.C,), torch.float32)
        return self._host

    def run_host(self, W_host, X_host, W_dev, X_dev, stream=None):
        """H2D copy of W and X, the path, D2H copy of codes / scales / npoints / points_used.
        Returns the host dict; the caller synchronizes ``stream`` before reading it."""
        st = stream or torch.cuda.current_stream()
        h = self.host_buffers()
        with torch.cuda.stream(st):
            W_dev.copy_(W_host, non_blocking=True)
            X_dev.copy_(X_host, non_blocking=True)
            self.run_device(W_dev, X_dev, stream=st)
            h["codes"].copy_(self.codes, non_blocking=True)
            h["scales"].copy_(self.scales, non_blocking=True)
            h["npoints"].copy_(self.npoints, non_blocking=True)
            h["points_used"].copy_(self.points_used, non_blocking=True)
            if self.center is not None:
                h["center"].copy_(self.center, non_blocking=True)
        return h

    def h2d_bytes(self, W, X) -> int:
        return W.numel() * W.element_size() + X.numel() * X.element_size()

    def d2h_bytes(self) -> int:
        s = self.spec
        return s.k_max * s.C * s.d + 4 * s.C * s.k_max + 4 * s.C + 4 + \
            (4 * s.C if self.center is not None else 0)


class NetworkPlan:
    """Every layer of a network through the path, layers spread over a pool of CUDA streams.

    Layers are independent (each has its own weights, calibration inputs and outputs), so their
    four-call chains run concurrently: small layers that cannot fill the GPU on their own overlap
    with the large ones.  Layers are issued largest first; the pool is forked from and joined back
    to the caller's stream, so the call as a whole is ordered like any single launch on it.
    """

    def __init__(self, specs, device, n_streams: int = 8, with_reconstruct: bool = True,
                 batch_alloc: bool = True):
        self.device = torch.device(device)
        # every layer's point counts in one buffer: [sum of C] npoints, then one total per layer
        # (one copy brings all of them back to the host)
        tot = sum(s.C for s in specs)
        self.counts = torch.empty((tot + len(specs),), dtype=torch.int32, device=self.device)
        self._counts_host = None
        offs = [0]
        for s in specs:
            offs.append(offs[-1] + s.C)
        self._count_views = [(offs[i], offs[i + 1], tot + i) for i in range(len(specs))]
        self.plans = [LayerPlan(s, self.device, with_reconstruct,
                                counts=(self.counts[a:b], self.counts[u:u + 1]))
                      for s, (a, b, u) in zip(specs, self._count_views)]
        # every layer's allocation in one launch (one CTA per layer) once all output errors are
        # in, instead of one single-CTA launch per layer -- where the layers share k_max and mode
        self.batch_alloc = (batch_alloc and len(specs) <= binding.MPQ_MAX_BATCH and
                            len({(s.k_max, s.mode) for s in specs}) == 1)
        work = [s.C * s.d * s.G * s.k_max + s.C * s.d * s.N for s in specs]
        self.order = sorted(range(len(specs)), key=lambda i: -work[i])
        self.streams = [torch.cuda.Stream(self.device) for _ in range(max(1, n_streams))]
        # host <-> device copies of run_host: one stream each way, so that no layer's input copy
        # waits in a compute stream's queue behind another layer's kernels
        self.copy_in = torch.cuda.Stream(self.device)
        self.copy_out = torch.cuda.Stream(self.device)

    def _fork(self, main):
        start = torch.cuda.Event()
        start.record(main)
        for s in self.streams:
            s.wait_event(start)

    def _join(self, main):
        for s in self.streams:
            e = torch.cuda.Event()
            e.record(s)
            main.wait_event(e)

    def run_device(self, Ws, Xs, stream=None, on_layer=None):
        """Ws[i], Xs[i]: device inputs of layer i.  on_layer(i, stream, phase), if given, is
        called around layer i's calls as LayerPlan.run_device's timing hook (phases 0..5)."""
        main = stream or torch.cuda.current_stream(self.device)
        self._fork(main)
        for n, i in enumerate(self.order):
            st = self.streams[n % len(self.streams)]
            hook = None if on_layer is None else (lambda ph, st=st, i=i: on_layer(i, st, ph))
            self.plans[i].run_device(Ws[i], Xs[i], stream=st, timing=hook,
                                     finish=not self.batch_alloc)
        self._join(main)
        if self.batch_alloc:
            self.allocate_all(main)
            self._fork(main)
            for n, i in enumerate(self.order):
                self.plans[i].run_reconstruct(self.streams[n % len(self.streams)])
            self._join(main)
        return self

    def allocate_all(self, stream):
        """Algorithm 2 for every layer in one launch (mpq_allocate_points_batched)."""
        p0 = self.plans[0].spec
        binding.mpq_allocate_points_batched([p.err for p in self.plans], p0.k_max, p0.mode,
                                            [p.spec.budget_or_eps for p in self.plans],
                                            npoints=[p.npoints for p in self.plans],
                                            points_used=[p.points_used for p in self.plans],
                                            stream=stream)

    def _host_counts(self):
        """Pinned host copy of the count buffer, and every plan's host views into it."""
        if self._counts_host is None:
            self._counts_host = torch.empty(self.counts.shape, dtype=torch.int32, pin_memory=True)
            for p, (a, b, u) in zip(self.plans, self._count_views):
                h = p.host_buffers(counts=(self._counts_host[a:b], self._counts_host[u:u + 1]))
                h["npoints"] = self._counts_host[a:b]            # also if made before
                h["points_used"] = self._counts_host[u:u + 1]
        return self._counts_host

    def _counts_out(self, p, h):
        with torch.cuda.stream(self.copy_out):
            h["npoints"].copy_(p.npoints, non_blocking=True)
            h["points_used"].copy_(p.points_used, non_blocking=True)
            if p.center is not None:
                h["center"].copy_(p.center, non_blocking=True)

    def run_host(self, W_hosts, X_hosts, W_devs, X_devs, stream=None, copy_inputs=True):
        """End to end: per layer, H2D of W and X from pinned memory, the path, D2H of codes,
        scales, point counts.  Input copies run back to back on one stream: every layer's W
        first, then every layer's X (largest layer first in both).  A layer's greedy search
        starts on its compute stream as soon as its W has landed and only its output error waits
        for its X, so the greedy searches overlap the calibration inputs' copies.  Outputs go
        back on one D2H stream: codes and scales as soon as the greedy search has made them
        (overlapping the layer's own output error and allocation), point counts once the
        allocation is done -- copies in both directions overlap kernels.  copy_inputs=False
        reuses the inputs an
        earlier call copied in (e.g. a second bit width over the same weights).  The caller
        synchronizes ``stream`` before reading the host outputs."""
        main = stream or torch.cuda.current_stream(self.device)
        counts_host = self._host_counts()
        self._fork(main)
        for s in (self.copy_in, self.copy_out):
            s.wait_stream(main)
        outs = [None] * len(self.plans)
        w_landed, x_landed = {}, {}
        with torch.cuda.stream(self.copy_in):
            for dst, src, landed in ((W_devs, W_hosts, w_landed), (X_devs, X_hosts, x_landed)):
                for i in self.order:
                    if copy_inputs:
                        dst[i].copy_(src[i], non_blocking=True)
                    landed[i] = torch.cuda.Event()
                    landed[i].record(self.copy_in)
        for n, i in enumerate(self.order):
            st = self.streams[n % len(self.streams)]
            st.wait_event(w_landed[i])
            p = self.plans[i]
            h = p.host_buffers()

            def points_out(phase, st=st, p=p, h=h):
                if phase != 2:            # after the greedy search: codes and scales are final
                    return
                made = torch.cuda.Event()
                made.record(st)
                self.copy_out.wait_event(made)
                with torch.cuda.stream(self.copy_out):
                    h["codes"].copy_(p.codes, non_blocking=True)
                    h["scales"].copy_(p.scales, non_blocking=True)

            p.run_device(W_devs[i], X_devs[i], stream=st, x_ready=x_landed[i], timing=points_out,
                         finish=not self.batch_alloc)
            outs[i] = h
            if self.batch_alloc:
                continue
            done = torch.cuda.Event()
            done.record(st)
            self.copy_out.wait_event(done)
            self._counts_out(p, h)
        self._join(main)
        if self.batch_alloc:
            self.allocate_all(main)
            done = torch.cuda.Event()
            done.record(main)
            self.copy_out.wait_event(done)
            with torch.cuda.stream(self.copy_out):   # every layer's counts in one copy
                counts_host.copy_(self.counts, non_blocking=True)
                for p, h in zip(self.plans, outs):
                    if p.center is not None:
                        h["center"].copy_(p.center, non_blocking=True)
            self._fork(main)
            for n, i in enumerate(self.order):
                self.plans[i].run_reconstruct(self.streams[n % len(self.streams)])
            self._join(main)
        for s in (self.copy_in, self.copy_out):
            e = torch.cuda.Event()
            e.record(s)
            main.wait_event(e)
        return outs


class CapturedNetwork:
    """A NetworkPlan's multi-stream step captured once into a CUDA graph and replayed.

    Capture records every launch of ``NetworkPlan.run_device`` (all layers, all streams, the fork and
    join) for fixed input tensors; each ``replay`` re-executes all of that work on the GPU with one
    host call.  Inputs are read from the captured tensors, so refresh their contents in place
    (``copy_``) to quantize new weights of the same shapes.  With ``host = (W_hosts, X_hosts)``
    (pinned) the captured step is ``NetworkPlan.run_host`` instead: every replay copies those host
    tensors in, runs the path and copies codes, scales and point counts out to the plans' pinned
    ``host_buffers()`` -- the end-to-end step for one host call (``copy_inputs=False``: the
    inputs are already on the device, only the outputs are copied out).
    """

    def __init__(self, net: NetworkPlan, Ws, Xs, warmup: int = 1, host=None,
                 copy_inputs: bool = True):
        self.net = net
        self.Ws, self.Xs = Ws, Xs
        self.host = host

        def step(st):
            if host is None:
                net.run_device(Ws, Xs, stream=st)
            else:
                net.run_host(host[0], host[1], Ws, Xs, stream=st, copy_inputs=copy_inputs)

        side = torch.cuda.Stream(net.device)
        side.wait_stream(torch.cuda.current_stream(net.device))
        with torch.cuda.stream(side):          # warm up outside capture (attributes, modules)
            for _ in range(warmup):
                step(side)
        torch.cuda.current_stream(net.device).wait_stream(side)
        torch.cuda.synchronize(net.device)
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=side):
            step(side)
        torch.cuda.synchronize(net.device)

    def replay(self):
        self.graph.replay()
        return self.net

    def host_outputs(self):
        """The pinned host outputs the end-to-end replays write (per layer)."""
        return [p.host_buffers() for p in self.net.plans]
