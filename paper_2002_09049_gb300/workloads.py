"""Seeded synthetic workloads: layer shapes, weight and calibration-input generators.

This module holds no arithmetic of the quantization method; it only draws inputs.  The CUDA path
(bench, tests) and the CPU oracle (tests, CPU baseline) both take their inputs from here, so they
always see the same numbers.

The paper quantizes pretrained ImageNet / VOC networks with 256 calibration images.  None of that
data is available, so five synthetic workloads with the same layer shapes stand in for it:

  c1  one conv-shaped layer 64 x 576, N(0, 2/576), X 512 x 576 ReLU(N(0,1))
  c2  ResNet-18 conv/fc shapes (21 layers), Kaiming normal N(0, 2/d), X 1024 x d ReLU(N(0,1))
  c3  ResNet-50 shapes (54 layers), heavy-tailed Student-t(4) rows scaled by lognormal(0, 0.5),
      X 2048 x d ReLU(N(0,1)); run at b = 4 and b = 3
  c4  MobileNetV2 shapes (53 layers, 17 depthwise 3x3 layers of d = 9), Laplace(0, 0.05),
      X 1024 x d ReLU(N(0,1)); depthwise layers get one 1024 x 9 block per channel
  c5  two large linear layers 4096 x 4096 and 11008 x 4096, N(0, 0.02^2) with 0.1 % of entries
      multiplied by 20, X 2048 x 4096 N(0,1) with 8 random columns multiplied by 10

Seeds: numpy Generator(PCG64(seed)); weights use seed 0 for c1 and 1000*config + layer index
otherwise; the calibration input of a layer uses the weight seed + 500000.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


@dataclass(frozen=True)
class Layer:
    name: str
    C: int          # output channels (rows of W)
    d: int          # weights per channel
    groups: int = 1  # 1: shared calibration input; C: one input block per channel (depthwise)


@dataclass(frozen=True)
class Workload:
    key: str
    title: str
    layers: tuple
    bits: tuple      # bit widths to run (c3 runs two)
    G: int           # candidate scales per step
    k_max: int       # points per channel
    beta: float      # average points per channel (budget)
    n_calib: int     # calibration rows per layer
    wdist: str
    xdist: str
    config_index: int
    extra: dict = field(default_factory=dict)

    @property
    def n_weights(self) -> int:
        return sum(l.C * l.d for l in self.layers)

    @property
    def n_channels(self) -> int:
        return sum(l.C for l in self.layers)

    def work_units(self, bits_runs: int | None = None) -> int:
        """Metric units of one pass: sum over layers of C * d * G * k_max (times the bit widths)."""
        runs = len(self.bits) if bits_runs is None else bits_runs
        return runs * sum(l.C * l.d for l in self.layers) * self.G * self.k_max


def _resnet18():
    L = [Layer("conv1", 64, 147)]
    for b in range(2):
        L += [Layer(f"layer1.{b}.conv1", 64, 576), Layer(f"layer1.{b}.conv2", 64, 576)]
    for stage, w in ((2, 128), (3, 256), (4, 512)):
        L += [Layer(f"layer{stage}.0.conv1", w, (w // 2) * 9),
              Layer(f"layer{stage}.0.conv2", w, w * 9),
              Layer(f"layer{stage}.0.downsample", w, w // 2),
              Layer(f"layer{stage}.1.conv1", w, w * 9),
              Layer(f"layer{stage}.1.conv2", w, w * 9)]
    L.append(Layer("fc", 1000, 512))
    return tuple(L)


def _resnet50():
    L = [Layer("conv1", 64, 147)]
    cin = 64
    for si, (w, nb) in enumerate(((64, 3), (128, 4), (256, 6), (512, 3)), start=1):
        for b in range(nb):
            L += [Layer(f"layer{si}.{b}.conv1", w, cin),
                  Layer(f"layer{si}.{b}.conv2", w, 9 * w),
                  Layer(f"layer{si}.{b}.conv3", 4 * w, w)]
            if b == 0:
                L.append(Layer(f"layer{si}.{b}.downsample", 4 * w, cin))
            cin = 4 * w
    L.append(Layer("fc", 1000, 2048))
    return tuple(L)


def _mobilenet_v2():
    L = [Layer("features.0", 32, 27)]
    cin = 32
    idx = 1
    for t, c, n, _s in ((1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2),
                        (6, 96, 3, 1), (6, 160, 3, 2), (6, 320, 1, 1)):
        for _ in range(n):
            h = cin * t
            if t != 1:
                L.append(Layer(f"features.{idx}.expand", h, cin))
            L.append(Layer(f"features.{idx}.dw", h, 9, groups=h))
            L.append(Layer(f"features.{idx}.project", c, h))
            cin = c
            idx += 1
    L.append(Layer("features.18", 1280, 320))
    L.append(Layer("classifier", 1000, 1280))
    return tuple(L)


WORKLOADS = {
    "c1": Workload("c1", "single conv-shaped layer 64x576", (Layer("conv", 64, 576),), (4,), 64, 4,
                   2.0, 512, "normal_fan_in", "relu_normal", 0),
    "c2": Workload("c2", "ResNet-18-shaped weight set", _resnet18(), (4,), 128, 4, 1.3, 1024,
                   "normal_fan_in", "relu_normal", 1),
    "c3": Workload("c3", "ResNet-50-shaped weight set, heavy-tailed", _resnet50(), (4, 3), 128, 6,
                   1.5, 2048, "student_t_lognormal", "relu_normal", 2),
    "c4": Workload("c4", "MobileNetV2-shaped weight set with depthwise 3x3", _mobilenet_v2(), (4,),
                   64, 8, 1.5, 1024, "laplace", "relu_normal", 3),
    "c5": Workload("c5", "large linear layers 4096x4096 and 11008x4096",
                   (Layer("q_proj", 4096, 4096), Layer("up_proj", 11008, 4096)), (4,), 256, 8, 1.25,
                   2048, "normal_outliers", "normal_hot_columns", 4),
}


def weight_seed(wl: Workload, layer_index: int) -> int:
    return 0 if wl.key == "c1" else 1000 * (wl.config_index + 1) + layer_index


def calib_seed(wl: Workload, layer_index: int) -> int:
    return weight_seed(wl, layer_index) + 500000


def make_weights(wl: Workload, layer_index: int, rows: tuple | None = None) -> np.ndarray:
    """C x d fp32 weight matrix of one layer (or the row range ``rows`` = (r0, r1) of it; the rows
    are the same numbers as in the full matrix)."""
    layer = wl.layers[layer_index]
    rng = np.random.Generator(np.random.PCG64(weight_seed(wl, layer_index)))
    C, d = layer.C, layer.d
    if wl.wdist == "normal_fan_in":
        W = rng.standard_normal((C, d)) * np.sqrt(2.0 / d)
    elif wl.wdist == "student_t_lognormal":
        nu = 4.0
        t = rng.standard_t(nu, size=(C, d)) * np.sqrt(2.0 / d) * np.sqrt((nu - 2.0) / nu)
        W = t * rng.lognormal(0.0, 0.5, size=(C, 1))
    elif wl.wdist == "laplace":
        W = rng.laplace(0.0, 0.05, size=(C, d))
    elif wl.wdist == "normal_outliers":
        W = rng.standard_normal((C, d)) * 0.02
        n_out = int(round(0.001 * C * d))
        pos = rng.choice(C * d, size=n_out, replace=False)
        W.reshape(-1)[pos] *= 20.0
    else:
        raise ValueError(wl.wdist)
    W = W.astype(np.float32)
    if rows is not None:
        W = W[rows[0]:rows[1]]
    return np.ascontiguousarray(W)


def make_calibration(wl: Workload, layer_index: int, n_rows: int | None = None,
                     channels: tuple | None = None) -> np.ndarray:
    """Calibration input of one layer: N x d fp32 (groups = 1) or C x N x d fp32 (depthwise).

    ``n_rows`` truncates to the first rows; ``channels`` = (c0, c1) selects depthwise blocks."""
    layer = wl.layers[layer_index]
    rng = np.random.Generator(np.random.PCG64(calib_seed(wl, layer_index)))
    N = wl.n_calib
    shape = (layer.C, N, layer.d) if layer.groups > 1 else (N, layer.d)
    if wl.xdist == "relu_normal":
        X = np.maximum(rng.standard_normal(shape), 0.0)
    elif wl.xdist == "normal_hot_columns":
        X = rng.standard_normal(shape)
        hot = rng.choice(layer.d, size=8, replace=False)
        X[..., hot] *= 10.0
    else:
        raise ValueError(wl.xdist)
    X = X.astype(np.float32)
    if layer.groups > 1 and channels is not None:
        X = X[channels[0]:channels[1]]
    if n_rows is not None:
        X = X[..., :n_rows, :]
    return np.ascontiguousarray(X)


def random_weights(C: int, d: int, seed: int, dist: str = "normal") -> np.ndarray:
    """Small ad-hoc test matrices (parity cases, edge cases)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    if dist == "normal":
        W = rng.standard_normal((C, d))
    elif dist == "laplace":
        W = rng.laplace(0.0, 1.0, size=(C, d))
    elif dist == "t":
        W = rng.standard_t(4.0, size=(C, d)) * rng.lognormal(0.0, 0.5, size=(C, 1))
    elif dist == "int":
        W = rng.integers(-7, 8, size=(C, d)).astype(np.float64) * 0.125
    else:
        raise ValueError(dist)
    return np.ascontiguousarray(W.astype(np.float32))


def random_calibration(N: int, d: int, seed: int, groups: int = 1) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    shape = (groups, N, d) if groups > 1 else (N, d)
    return np.ascontiguousarray(np.maximum(rng.standard_normal(shape), 0.0).astype(np.float32))
