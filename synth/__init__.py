"""Seeded synthetic workloads for the fused-tile CNN front-end.

This module holds only data: the layer lists of the workloads, their plan
parameters, and seeded random tensors.  It contains none of the method's
arithmetic (no convolution, no region or memory computation), so both the
CPU oracle and the CUDA path can take their inputs from it without sharing
any code with each other.

Layer tuples are ``(type, k, stride, pad, filters)`` with type ``"conv"`` or
``"max"``; ``filters`` is ignored for max-pool layers.  The YOLOv2 front-end is
the first 16 layers of YOLOv2 that the paper evaluates (Sec. 2); the random
distributions are those of the tiny three-layer workload (uniform inputs,
He-normal weights, folded batch-norm scale/bias, leaky ReLU 0.1).
"""
from __future__ import annotations

import numpy as np

CONV = "conv"
MAX = "max"

# YOLOv2 first 16 layers (Sec. 2): 3x3 convs pad 1, 1x1 convs pad 0, 2x2/s2 pools.
YOLO16 = [
    (CONV, 3, 1, 1, 32),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 64),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 128),
    (CONV, 1, 1, 0, 64),
    (CONV, 3, 1, 1, 128),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 256),
    (CONV, 1, 1, 0, 128),
    (CONV, 3, 1, 1, 256),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 512),
    (CONV, 1, 1, 0, 256),
    (CONV, 3, 1, 1, 512),
    (CONV, 1, 1, 0, 256),
]

# The rest of the YOLOv2 trunk up to its route layer: conv 3x3 512, max-pool, then at 1/32
# resolution conv 3x3 1024, 1x1 512, 3x3 1024, 1x1 512, 3x3 1024 and two detection-head
# 3x3 1024 convolutions (25 layers in all; every later layer is a route, reorg or concat).
YOLO25 = YOLO16 + [
    (CONV, 3, 1, 1, 512),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 1024),
    (CONV, 1, 1, 0, 512),
    (CONV, 3, 1, 1, 1024),
    (CONV, 1, 1, 0, 512),
    (CONV, 3, 1, 1, 1024),
    (CONV, 3, 1, 1, 1024),
    (CONV, 3, 1, 1, 1024),
]

# Tiny three-layer stack used for fp32 parity.
TINY3 = [
    (CONV, 3, 1, 1, 8),
    (MAX, 2, 2, 0, 0),
    (CONV, 3, 1, 1, 16),
]

SEED_BASE = 2107069600

# Workloads.  ``cut`` is the paper's cut: the index of the first layer of the
# second group (Sec. 4), or None for a single group.  Grids are (N, M) tiles
# along (rows, cols) of each group's last-layer output.
WORKLOADS = {
    "tiny3_64_fp32": dict(layers=TINY3, h=64, w=64, c=3, batch=1, dtype="fp32",
                          cut=None, grids=[(2, 2)], seed=SEED_BASE + 0),
    "yolo16_416_1x3x3": dict(layers=YOLO16, h=416, w=416, c=3, batch=1, dtype="bf16",
                             cut=None, grids=[(3, 3)], seed=SEED_BASE + 1),
    "yolo16_608_5x5_c8_2x2": dict(layers=YOLO16, h=608, w=608, c=3, batch=1, dtype="bf16",
                                  cut=8, grids=[(5, 5), (2, 2)], seed=SEED_BASE + 2),
    "yolo16_1216_b8_8x8_c8_4x4": dict(layers=YOLO16, h=1216, w=1216, c=3, batch=8, dtype="bf16",
                                      cut=8, grids=[(8, 8), (4, 4)], seed=SEED_BASE + 4),
    # a second workload: the whole YOLOv2 trunk (weight-heavy 1024-channel layers at 19x19)
    "yolo25_96_2x2_c8_1x1": dict(layers=YOLO25, h=96, w=96, c=3, batch=2, dtype="bf16",
                                 cut=8, grids=[(2, 2), (1, 1)], seed=SEED_BASE + 5),
    "yolo25_608_5x5_c8_2x2": dict(layers=YOLO25, h=608, w=608, c=3, batch=1, dtype="bf16",
                                  cut=8, grids=[(5, 5), (2, 2)], seed=SEED_BASE + 6),
}
# The sweep: cut after layer 1, 3, 7, 11 (paper cut 2, 4, 8, 12) x grids 1..5 per group.
SWEEP_CUTS = [2, 4, 8, 12]
SWEEP_GRIDS = [1, 2, 3, 4, 5]
SWEEP_SEED = SEED_BASE + 3


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), kept as float32.

    A data-representation step applied once when inputs are generated, so that
    both sides consume exactly the same values.
    """
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out = out.copy()
        out[nan] = np.nan
    return out


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """Upper 16 bits of float32 values that are already bf16-representable."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    return (a.view(np.uint32) >> 16).astype(np.uint16)


def layer_channels(layers, c_in):
    """Input channel count of every layer (plain bookkeeping of the list)."""
    cs = []
    c = c_in
    for (t, k, s, p, f) in layers:
        cs.append(c)
        if t == CONV:
            c = f
    return cs


def make_params(layers, c_in, seed, dtype="bf16"):
    """Seeded per-layer parameters.

    Returns a list with, for each layer, None (max-pool) or a tuple
    ``(w[Cout][Cin][k][k], scale[Cout], bias[Cout])`` of float32 arrays.
    w ~ N(0, 2/fan_in) (He-normal, fan_in = Cin*k*k), scale ~ U[0.5, 1.5),
    bias ~ N(0, 0.1^2).  In bf16 mode the weights are rounded to bf16 once;
    scale and bias stay float32.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    cs = layer_channels(layers, c_in)
    params = []
    for (t, k, s, p, f), cin in zip(layers, cs):
        if t != CONV:
            params.append(None)
            continue
        fan_in = cin * k * k
        w = rng.standard_normal((f, cin, k, k)).astype(np.float32) * np.float32(np.sqrt(2.0 / fan_in))
        scale = rng.uniform(0.5, 1.5, size=f).astype(np.float32)
        bias = (rng.standard_normal(f) * 0.1).astype(np.float32)
        if dtype == "bf16":
            w = round_bf16(w)
        params.append((np.ascontiguousarray(w), scale, bias))
    return params


def make_input(batch, h, w, c, seed, dtype="bf16"):
    """Seeded input images [B][H][W][C], uniform on [0, 1), float32 (bf16-rounded in bf16 mode)."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    x = rng.random((batch, h, w, c), dtype=np.float32)
    if dtype == "bf16":
        x = round_bf16(x)
    return np.ascontiguousarray(x)


def workload(name):
    """Layers, params and input of a named workload."""
    wl = dict(WORKLOADS[name])
    wl["params"] = make_params(wl["layers"], wl["c"], wl["seed"], wl["dtype"])
    wl["input"] = make_input(wl["batch"], wl["h"], wl["w"], wl["c"], wl["seed"], wl["dtype"])
    return wl
