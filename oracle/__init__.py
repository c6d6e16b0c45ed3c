"""The oracle: a plain, slow, obviously correct CPU implementation of MAFAT's hot path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product package imports, loads or
calls this package; only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA path; the two meet only in the seeded inputs of
``synth``.

Contents, each following the paper (MAFAT, arXiv 2107.06960):

* ``layer_shapes``      -- shape inference of conv / max-pool layers (Sec. 4.1,
                           the W, H, F, S network description).
* ``grid_bounds``       -- the even N x M partition of a group's output (Sec. 4).
* ``tile_regions``      -- the ``Grid`` back-traversal of a tile through its
                           group (Sec. 4.1, FTP of Sec. 3).
* ``predict_layer_group`` / ``predict_mem`` -- the memory predictor (Algorithm 1).
* ``get_config``        -- the configuration search (Algorithm 2).
* ``forward``           -- layer-by-layer fp64 forward (the plain definition); the
                           same loops in fp32 (``precision="f32"``) are the timed CPU
                           baseline.
* ``forward_tiled``     -- the same network executed as fused tiles of its layer
                           groups, merged and re-tiled at every cut (Sec. 4).

Readings of passages that are garbled or silent are stated where they are used.
Parity of the predictor's absolute values beyond its units is unpinned (the
paper's 66 MB figure for 5x5/8/2x2 is not reproduced by the literal algorithm).
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build import LIB, LIB_F32, build_oracle

CONV = "conv"
MAX = "max"
LEAKY_SLOPE = 0.1
BIAS_MIB = 31.0          # Sec. 4.1: constant bias term of 31 MB
BYTES_PER_ELEM = 4       # fp32 elements (Darknet); pinned by the 100 MB / 135 MB figures of Sec. 2

_libs = {}
_CT = {"f64": (ctypes.c_double, np.float64), "f32": (ctypes.c_float, np.float32)}


def _load(precision="f64"):
    """The oracle's C library: "f64" (the parity oracle) or "f32" (the same loops in
    single precision, the CPU baseline the benchmark times)."""
    if precision not in _libs:
        build_oracle()
        lib = ctypes.CDLL(LIB if precision == "f64" else LIB_F32)
        real = _CT[precision][0]
        dp = ctypes.POINTER(real)
        i = ctypes.c_int
        lib.oracle_conv_full.argtypes = [dp, i, i, i, dp, i, i, i, i, dp, dp, real, dp]
        lib.oracle_maxpool_full.argtypes = [dp, i, i, i, i, i, dp]
        lib.oracle_conv_region.argtypes = [dp, i, i, i, i, i, i, i, dp, i, i, i, i, dp, dp,
                                           real, i, i, i, i, dp]
        lib.oracle_maxpool_region.argtypes = [dp, i, i, i, i, i, i, i, i, i, i, i, i, i, dp]
        for f in (lib.oracle_conv_full, lib.oracle_maxpool_full, lib.oracle_conv_region,
                  lib.oracle_maxpool_region):
            f.restype = ctypes.c_int
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_set_num_threads.argtypes = [i]
        lib.oracle_set_num_threads.restype = None
        _libs[precision] = lib
    return _libs[precision]


def _dp(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def num_threads(precision="f64"):
    return _load(precision).oracle_num_threads()


def set_num_threads(n, precision="f64"):
    """OpenMP threads of the oracle's loops (n >= 1)."""
    _load(precision).oracle_set_num_threads(int(n))


# ---------------------------------------------------------------------------
# Network description and tiling (Sec. 4, Sec. 4.1)
# ---------------------------------------------------------------------------

def layer_shapes(layers, h, w, c):
    """Shape inference: out = floor((in + 2p - k) / s) + 1 per layer.

    Returns a list of dicts with in/out height, width and channels of every
    layer; a max-pool keeps the channel count, a conv produces ``filters``.
    """
    shapes = []
    for (t, k, s, p, f) in layers:
        oh = (h + 2 * p - k) // s + 1
        ow = (w + 2 * p - k) // s + 1
        oc = f if t == CONV else c
        shapes.append(dict(h_in=h, w_in=w, c_in=c, h_out=oh, w_out=ow, c_out=oc))
        h, w, c = oh, ow, oc
    return shapes


def groups_of(n_layers, cut):
    """Layer groups for a cut (Sec. 4): group 1 is layers 0..cut-1, group 2 is
    cut..n-1.  The paper writes "to layer n"; with 0-based layers that is n-1.
    A cut of None (or n, the paper's "16" / NoCut) means a single group.  A list
    of increasing cuts gives more groups the same way (the paper uses at most
    two; more is the generalisation its Sec. 6 points to)."""
    if cut is None or (not isinstance(cut, (list, tuple)) and cut >= n_layers):
        return [(0, n_layers - 1)]
    cuts = list(cut) if isinstance(cut, (list, tuple)) else [cut]
    if any(c <= 0 or c >= n_layers for c in cuts) or any(a >= b for a, b in zip(cuts, cuts[1:])):
        raise ValueError("cuts must increase within 1..n-1")
    bounds = [0] + cuts + [n_layers]
    return [(a, b - 1) for a, b in zip(bounds, bounds[1:])]


def grid_bounds(length, n):
    """Even partition of ``length`` into ``n`` parts: part i is
    [floor(i*L/n), floor((i+1)*L/n)).  (The paper says only "even"; any
    partition gives the same output.)"""
    return [(i * length // n, (i + 1) * length // n) for i in range(n)]


def _back(rng, k, s, p, size_in):
    """Input interval of a layer needed for output interval [a, b): the window
    of output a starts at a*s - p, that of output b-1 ends at (b-1)*s - p + k - 1;
    clipped to the map (zero padding lies outside it)."""
    a, b = rng
    if b <= a:
        return (0, 0)
    lo = a * s - p
    hi = (b - 1) * s - p + k
    return (max(lo, 0), min(hi, size_in))


def tile_regions(layers, shapes, group, n, m, i, j, bounds=None):
    """The ``Grid`` traversal: for tile (i, j) of an n x m grid on the group's
    last-layer output, the output and input rectangle of every layer of the
    group, walking from the last layer back to the first.  ``bounds`` = (row
    bounds, column bounds) gives a non-uniform grid (n + 1 and m + 1 increasing
    values from 0 to the map size); None means the even grid.

    Returns {layer: (out_rect, in_rect)} with rect = (y0, y1, x0, x1), half-open.
    """
    first, last = group
    sh = shapes[last]
    if bounds is None:
        rows = grid_bounds(sh["h_out"], n)[i]
        cols = grid_bounds(sh["w_out"], m)[j]
    else:
        rb, cb = bounds
        for b, size, parts in ((rb, sh["h_out"], n), (cb, sh["w_out"], m)):
            if len(b) != parts + 1 or b[0] != 0 or b[-1] != size or any(x >= y for x, y in zip(b, b[1:])):
                raise ValueError("tile bounds do not partition the group output")
        rows, cols = (rb[i], rb[i + 1]), (cb[j], cb[j + 1])
    out = {}
    for l in range(last, first - 1, -1):
        t, k, s, p, f = layers[l]
        iy = _back(rows, k, s, p, shapes[l]["h_in"])
        ix = _back(cols, k, s, p, shapes[l]["w_in"])
        out[l] = ((rows[0], rows[1], cols[0], cols[1]), (iy[0], iy[1], ix[0], ix[1]))
        rows, cols = iy, ix
    return out


# ---------------------------------------------------------------------------
# Memory predictor (Algorithm 1) and configuration search (Algorithm 2)
# ---------------------------------------------------------------------------

def layer_group_terms(layers, shapes, group, n, m, i, j, l):
    """The three sizes Algorithm 1 computes for tile (i, j) at layer l, in
    elements: scratch = w_out*h_out*c_in*F^2/S, input = w_in*h_in*c_in,
    output = w_out*h_out*c_out, with the tile's w/h in/out from the Grid
    traversal (tile_regions) and c_in, c_out the layer's channel counts."""
    t, k, s, p, f = layers[l]
    (oy0, oy1, ox0, ox1), (iy0, iy1, ix0, ix1) = tile_regions(layers, shapes, group, n, m, i, j)[l]
    w_out, h_out = ox1 - ox0, oy1 - oy0
    w_in, h_in = ix1 - ix0, iy1 - iy0
    c_in, c_out = shapes[l]["c_in"], shapes[l]["c_out"]
    scratch = w_out * h_out * c_in * (k * k) / s
    inp = w_in * h_in * c_in
    outp = w_out * h_out * c_out
    return scratch, inp, outp


def predict_layer_group(layers, shapes, group, n, m, bias_mib=BIAS_MIB,
                        input_factor=2, bytes_per_elem=BYTES_PER_ELEM):
    """Algorithm 1, literal reading: the maximum over tiles (i, j) of the grid
    and over the layers of the group of scratch + output + 2*input (the terms
    of layer_group_terms), converted from elements to MiB, plus the bias.  The
    printed loop ``l <- bottom; while l <= top; l <- l - 1`` is read as visiting
    every layer of the group once (the order does not matter to a maximum);
    ``for i in 0..N`` is read as i = 0..N-1."""
    first, last = group
    best = 0.0
    for i in range(n):
        for j in range(m):
            for l in range(first, last + 1):
                scratch, inp, outp = layer_group_terms(layers, shapes, group, n, m, i, j, l)
                mem = scratch + outp + inp * input_factor
                if mem > best:
                    best = mem
    return best * bytes_per_elem / float(1 << 20) + bias_mib


def predict_mem(layers, shapes, cut, grids, bias_mib=BIAS_MIB, input_factor=2):
    """Prediction of a whole configuration: the maximum over its layer groups
    (Sec. 4.1).  ``grids`` gives (N, M) per group."""
    gs = groups_of(len(layers), cut)
    return max(predict_layer_group(layers, shapes, g, nm[0], nm[1], bias_mib, input_factor)
               for g, nm in zip(gs, grids))


def get_config(layers, shapes, limit_mib, predictor=None, cuts=None, tiles=(1, 2, 3, 4, 5),
               bottom_tile=2, bias_mib=BIAS_MIB):
    """Algorithm 2: greedy search over cut in {n (no cut), 12, 8} and square
    top tilings 1..5 with a 2x2 bottom tiling; returns the first configuration
    whose prediction is strictly below the limit, else the configuration the
    loops end on (5x5 / cut 8 / 2x2).

    Readings: the printed ``LG_2 <- 4`` contradicts the text and Table 1
    (the bottom tiling is always 2x2), so the bottom tiling is 2x2; the
    unused ``getMaxLayer`` line is dropped.  ``predictor(cut, n1, n2)`` may be
    supplied to exercise the control flow alone.

    Returns (top_tile, bottom_tile, cut) with cut == n meaning NoCut.
    """
    n = len(layers)
    if cuts is None:
        cuts = (n, 12, 8)
    if predictor is None:
        def predictor(cut, t1, t2):
            grids = [(t1, t1)] if cut >= n else [(t1, t1), (t2, t2)]
            return predict_mem(layers, shapes, None if cut >= n else cut, grids, bias_mib)
    lg1, cut = None, None
    for cut in cuts:
        for tile in tiles:
            lg1 = tile
            if predictor(cut, lg1, bottom_tile) < limit_mib:
                return lg1, bottom_tile, cut
    return lg1, bottom_tile, cut


# ---------------------------------------------------------------------------
# Forward passes (fp64)
# ---------------------------------------------------------------------------

def _ptr(a, precision):
    return a.ctypes.data_as(ctypes.POINTER(_CT[precision][0]))


def _conv_full(x, prm, k, s, p, precision="f64"):
    w, scale, bias = prm
    H, W, C = x.shape
    Cout = w.shape[0]
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    dt = _CT[precision][1]
    out = np.empty((Ho, Wo, Cout), dtype=dt)
    xx = np.ascontiguousarray(x, dtype=dt)
    ww = np.ascontiguousarray(w, dtype=dt)
    sc = np.ascontiguousarray(scale, dtype=dt)
    bi = np.ascontiguousarray(bias, dtype=dt)
    q = lambda a: _ptr(a, precision)
    rc = _load(precision).oracle_conv_full(q(xx), H, W, C, q(ww), Cout, k, s, p, q(sc), q(bi),
                                           LEAKY_SLOPE, q(out))
    if rc != 0:
        raise ValueError("oracle_conv_full: bad sizes")
    return out


def _pool_full(x, k, s, precision="f64"):
    H, W, C = x.shape
    Ho, Wo = (H - k) // s + 1, (W - k) // s + 1
    dt = _CT[precision][1]
    out = np.empty((Ho, Wo, C), dtype=dt)
    xx = np.ascontiguousarray(x, dtype=dt)
    if _load(precision).oracle_maxpool_full(_ptr(xx, precision), H, W, C, k, s, _ptr(out, precision)) != 0:
        raise ValueError("oracle_maxpool_full: bad sizes")
    return out


def apply_layer(layer, prm, x, precision="f64"):
    """One layer on a full HWC map (fp64, or fp32 with precision="f32")."""
    t, k, s, p, f = layer
    if t == CONV:
        return _conv_full(x, prm, k, s, p, precision)
    return _pool_full(x, k, s, precision)


def forward(layers, params, x, precision="f64"):
    """Layer-by-layer forward of one HWC image; returns the list of every layer's output.
    precision="f32" runs the same loops in single precision (every sum and every layer
    output in fp32): the plain fp32 forward used as the timed CPU baseline."""
    outs = []
    cur = np.asarray(x, dtype=_CT[precision][1])
    for layer, prm in zip(layers, params):
        cur = apply_layer(layer, prm, cur, precision)
        outs.append(cur)
    return outs


def group_outputs(layers, params, x, cut):
    """Outputs of each layer group (the cut tensors, then the final output) of one image."""
    outs = forward(layers, params, x)
    return [outs[last] for (first, last) in groups_of(len(layers), cut)]


def _region_layer(layer, prm, buf, in_rect, map_hw, out_rect):
    t, k, s, p, f = layer
    iy0, iy1, ix0, ix1 = in_rect
    oy0, oy1, ox0, ox1 = out_rect
    mh, mw = map_hw
    C = buf.shape[2]
    xx = np.ascontiguousarray(buf, dtype=np.float64)
    lib = _load()
    if t == CONV:
        w, scale, bias = prm
        Cout = w.shape[0]
        out = np.empty((oy1 - oy0, ox1 - ox0, Cout), dtype=np.float64)
        ww = np.ascontiguousarray(w, dtype=np.float64)
        sc = np.ascontiguousarray(scale, dtype=np.float64)
        bi = np.ascontiguousarray(bias, dtype=np.float64)
        rc = lib.oracle_conv_region(_dp(xx), iy0, ix0, iy1 - iy0, ix1 - ix0, mh, mw, C, _dp(ww), Cout,
                                    k, s, p, _dp(sc), _dp(bi), LEAKY_SLOPE,
                                    oy0, ox0, oy1 - oy0, ox1 - ox0, _dp(out))
    else:
        out = np.empty((oy1 - oy0, ox1 - ox0, C), dtype=np.float64)
        rc = lib.oracle_maxpool_region(_dp(xx), iy0, ix0, iy1 - iy0, ix1 - ix0, mh, mw, C, k, s,
                                       oy0, ox0, oy1 - oy0, ox1 - ox0, _dp(out))
    if rc != 0:
        raise RuntimeError("tile region is missing input it needs")
    return out


def forward_tiled(layers, params, x, cut, grids, bounds=None):
    """Fused tile partitioning of the layer groups of ``cut`` (Sec. 3, Sec. 4).

    Each group's last-layer output is split into an N x M grid; every tile
    runs all layers of its group on its own regions (recomputing the overlap),
    and writes its rectangle of the group output.  The next group re-tiles the merged
    cut tensor.  ``bounds`` (one (row bounds, column bounds) pair per group, or
    None) gives non-uniform grids.  Returns the group outputs; raises if the
    tiles do not cover the group output exactly once.
    """
    shapes = layer_shapes(layers, x.shape[0], x.shape[1], x.shape[2])
    gin = np.asarray(x, dtype=np.float64)
    results = []
    for gi, (g, (n, m)) in enumerate(zip(groups_of(len(layers), cut), grids)):
        gb = None if bounds is None else bounds[gi]
        first, last = g
        sh = shapes[last]
        gout = np.zeros((sh["h_out"], sh["w_out"], sh["c_out"]), dtype=np.float64)
        cover = np.zeros((sh["h_out"], sh["w_out"]), dtype=np.int64)
        for i in range(n):
            for j in range(m):
                regs = tile_regions(layers, shapes, g, n, m, i, j, gb)
                out_rect_last = regs[last][0]
                if out_rect_last[1] <= out_rect_last[0] or out_rect_last[3] <= out_rect_last[2]:
                    continue
                iy0, iy1, ix0, ix1 = regs[first][1]
                buf = gin[iy0:iy1, ix0:ix1, :]
                in_rect = regs[first][1]
                for l in range(first, last + 1):
                    out_rect, in_rect_l = regs[l]
                    assert in_rect_l == in_rect
                    buf = _region_layer(layers[l], params[l], buf, in_rect,
                                        (shapes[l]["h_in"], shapes[l]["w_in"]), out_rect)
                    in_rect = out_rect
                oy0, oy1, ox0, ox1 = out_rect_last
                gout[oy0:oy1, ox0:ox1, :] = buf
                cover[oy0:oy1, ox0:ox1] += 1
        if not np.all(cover == 1):
            raise RuntimeError("tiles do not partition the group output")
        results.append(gout)
        gin = gout
    return results


def conv_flops(layers, shapes):
    """Useful multiply-add work of the convs, in FLOPs (2 per MAC), per image."""
    tot = 0
    for (t, k, s, p, f), sh in zip(layers, shapes):
        if t == CONV:
            tot += 2 * sh["h_out"] * sh["w_out"] * sh["c_out"] * sh["c_in"] * k * k
    return tot
