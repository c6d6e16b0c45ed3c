"""GB300-native fused-tile execution of CNN layer groups (MAFAT, arXiv 2107.06960).

A thin ctypes binding of ``libmafat.so`` (the C ABI declared in
``include/mafat.h``): it only marshals arguments.  Every step of the hot path
runs in the library's CUDA kernels; there is no CPU fallback, and importing
this package fails loudly when the library has not been built
(``python -c "import __graft_entry__ as g; g.build()"``).

Names follow the paper: a network is a list of conv / max-pool layers; a plan
cuts it into at most two layer groups (``cut`` = first layer of group 2) and
tiles each group's output with an N x M grid.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmafat.so")

MAFAT_CONV, MAFAT_MAXPOOL = 0, 1
BF16, FP32 = 0, 1
STATUS = {0: "OK", 1: "EINVAL", 2: "EUNSUPPORTED", 3: "ENOMEM", 4: "ECUDA", 5: "ETIMEOUT", 6: "ENOFIT",
          7: "EDEVICE"}
OK, EINVAL, EUNSUPPORTED, ENOMEM, ECUDA, ETIMEOUT, ENOFIT, EDEVICE = range(8)

i32, i64, dbl, vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p


class LayerDesc(ctypes.Structure):
    _fields_ = [("type", i32), ("k", i32), ("stride", i32), ("pad", i32), ("filters", i32)]


class PlanOptions(ctypes.Structure):
    _fields_ = [("struct_size", i32), ("ring_slots", i32), ("wave_tiles", i32), ("max_ctas", i32),
                ("wait_timeout_ns", i64), ("test_unpublished_task", i32), ("dry_run", i32),
                ("trace", i32), ("force_nblk", i32), ("force_mb", i32), ("lookahead_items", i32),
                ("tile_bounds", ctypes.POINTER(i32)), ("halo_reuse", i32), ("frame_major", i32),
                ("chain", i32), ("rect_blocks", i32)]


class PlanStats(ctypes.Structure):
    _fields_ = [("struct_size", i32), ("n_groups", i32), ("n_tiles", i32), ("n_tasks", i32),
                ("n_items", i64), ("useful_flops", dbl), ("executed_flops", dbl), ("issued_flops", dbl),
                ("predicted_mib", dbl), ("group_io_bytes", i64), ("weight_bytes", i64),
                ("scratch_bytes", i64), ("workspace_bytes", i64), ("smem_bytes_per_cta", i64),
                ("ring_slots", i32), ("wave_tiles", i32), ("max_ctas", i32), ("dtype", i32),
                ("frames_overlapped", i32), ("reserved", i32)]


class SearchOptions(ctypes.Structure):
    _fields_ = [("struct_size", i32), ("batch", i32), ("dtype", i32), ("include_one_group", i32),
                ("n_cuts", i32), ("cuts", ctypes.POINTER(i32)), ("max_grid", i32), ("square_only", i32),
                ("budget_bytes", i64), ("runs", i32), ("flush_l2", i32), ("dry_run", i32),
                ("reserved", i32 * 3)]


class SearchCandidate(ctypes.Structure):
    _fields_ = [("n_groups", i32), ("cut", i32), ("grid_n", i32 * 2), ("grid_m", i32 * 2),
                ("intermediate_bytes", i64), ("predicted_mib", dbl), ("executed_flops", dbl),
                ("us_per_run", dbl), ("status", i32), ("reserved", i32)]


# (name, restype, argtypes) of every entry point of include/mafat.h
_SIGNATURES = [
    ("mafat_describe_net", i32, [vp, i32, i32, i32, i32, ctypes.POINTER(vp)]),
    ("mafat_net_shape", i32, [vp, i32, ctypes.POINTER(i32)]),
    ("mafat_set_weights", i32, [vp, i32, vp, vp, vp]),
    ("mafat_plan", i32, [vp, i32, ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32), i32, i32,
                         ctypes.POINTER(vp)]),
    ("mafat_plan_ex", i32, [vp, i32, ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32), i32, i32,
                            ctypes.POINTER(PlanOptions), ctypes.POINTER(vp)]),
    ("mafat_run", i32, [vp, vp, vp, vp]),
    ("mafat_run_debug", i32, [vp, vp, vp, vp, vp]),
    ("mafat_run_host", i32, [vp, vp, vp, vp]),
    ("mafat_run_host_async", i32, [vp, vp, vp, vp]),
    ("mafat_run_host_wait", i32, [vp]),
    ("mafat_sync_status", i32, [vp, vp]),
    ("mafat_tile_region", i32, [vp, i32, i32, i32, i32, ctypes.POINTER(i32), ctypes.POINTER(i32)]),
    ("mafat_net_tile_region", i32, [vp, i32, i32, i32, i32, i32, i32, i32, ctypes.POINTER(i32),
                                    ctypes.POINTER(i32)]),
    ("mafat_predict_layer_group", i32, [vp, i32, i32, i32, i32, dbl, i32, ctypes.POINTER(dbl)]),
    ("mafat_predict_mem", i32, [vp, i32, i32, i32, i32, i32, dbl, ctypes.POINTER(dbl)]),
    ("mafat_search", i32, [vp, dbl, dbl, ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32)]),
    ("mafat_balanced_bounds", i32, [vp, i32, i32, i32, i32, ctypes.POINTER(i32), ctypes.POINTER(i32)]),
    ("mafat_plan_stats", i32, [vp, ctypes.POINTER(PlanStats)]),
    ("mafat_search_measured", i32, [vp, ctypes.POINTER(SearchOptions), vp, ctypes.POINTER(SearchCandidate), i32,
                                    ctypes.POINTER(i32), ctypes.POINTER(i32)]),
    ("mafat_launches_per_run", i32, [vp]),
    ("mafat_plan_trace", i32, [vp, vp, i64, vp]),
    ("mafat_plan_destroy", None, [vp]),
    ("mafat_net_destroy", None, [vp]),
    ("mafat_last_error", ctypes.c_char_p, []),
    ("mafat_version", ctypes.c_char_p, []),
    ("mafat_diag_umma", i32, [vp, vp, vp, i32, i32, vp]),
    ("mafat_run_fp32_noalloc", i32, [vp, vp, vp, vp]),
    ("mafat_noalloc_sync_status", i32, [vp]),
]
EXPORTED = [s[0] for s in _SIGNATURES]

if not os.path.exists(LIB_PATH):
    raise ImportError("libmafat.so is not built (expected at %s); build it with "
                      "paper_2107_06960_gb300.build.build()" % LIB_PATH)
lib = ctypes.CDLL(LIB_PATH)
for _name, _res, _args in _SIGNATURES:
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args


class MafatError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s: %s" % (STATUS.get(status, status), msg))
        self.status = status


def _check(status):
    if status != 0:
        raise MafatError(status, lib.mafat_last_error().decode())


def _ptr(x):
    """Device/host address of a tensor (anything with data_ptr()), a numpy array, or an int."""
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    return int(x)


def _stream(stream, like=None):
    if stream is not None:
        return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    if like is not None and getattr(like, "is_cuda", False):
        import torch
        return torch.cuda.current_stream(like.device).cuda_stream
    return None


def _rect():
    return (i32 * 4)()


def layer_descs(layers):
    """Layer tuples ("conv"|"max", k, stride, pad, filters) -> LayerDesc array."""
    arr = (LayerDesc * len(layers))()
    for d, (t, k, s, p, f) in zip(arr, layers):
        d.type = MAFAT_CONV if t == "conv" else MAFAT_MAXPOOL
        d.k, d.stride, d.pad, d.filters = k, s, p, f
    return arr


class Net:
    """mafat_describe_net / mafat_set_weights and the host-side planner queries."""

    def __init__(self, layers, h, w, c):
        self.layers = list(layers)
        self._descs = layer_descs(self.layers)
        h_ = vp()
        _check(lib.mafat_describe_net(ctypes.cast(self._descs, vp), len(self.layers), h, w, c, ctypes.byref(h_)))
        self.handle = h_

    def shape(self, layer):
        s = (i32 * 6)()
        _check(lib.mafat_net_shape(self.handle, layer, s))
        return tuple(s)

    def set_weights(self, layer, w, scale, bias):
        import numpy as np
        w = np.ascontiguousarray(w, dtype=np.float32)
        scale = np.ascontiguousarray(scale, dtype=np.float32)
        bias = np.ascontiguousarray(bias, dtype=np.float32)
        _check(lib.mafat_set_weights(self.handle, layer, w.ctypes.data, scale.ctypes.data, bias.ctypes.data))

    def set_params(self, params):
        for l, prm in enumerate(params):
            if prm is not None:
                self.set_weights(l, *prm)

    def tile_region(self, first, last, n, m, i, j, layer):
        a, b = _rect(), _rect()
        _check(lib.mafat_net_tile_region(self.handle, first, last, n, m, i, j, layer, a, b))
        return tuple(b), tuple(a)  # (out_rect, in_rect)

    def predict_layer_group(self, first, last, n, m, bias_mib=31.0, input_factor=2):
        out = dbl()
        _check(lib.mafat_predict_layer_group(self.handle, first, last, n, m, bias_mib, input_factor,
                                             ctypes.byref(out)))
        return out.value

    def predict_mem(self, cut, n1, m1, n2, m2, bias_mib=31.0):
        out = dbl()
        _check(lib.mafat_predict_mem(self.handle, cut, n1, m1, n2, m2, bias_mib, ctypes.byref(out)))
        return out.value

    def search(self, limit_mib, bias_mib=31.0):
        a, c, b = i32(), i32(), i32()
        _check(lib.mafat_search(self.handle, limit_mib, bias_mib, ctypes.byref(a), ctypes.byref(c), ctypes.byref(b)))
        return a.value, b.value, c.value  # (top_tile, bottom_tile, cut)

    def balanced_bounds(self, first, last, n, m):
        """Work-balanced non-uniform tile bounds (rows, cols) of an n x m grid on the output of
        layers first..last (mafat_balanced_bounds)."""
        r, c = (i32 * (n + 1))(), (i32 * (m + 1))()
        _check(lib.mafat_balanced_bounds(self.handle, first, last, n, m, r, c))
        return list(r), list(c)

    def search_measured(self, cuts=(2, 4, 8, 12), include_one_group=True, max_grid=5, square_only=True,
                        budget_bytes=0, runs=10, flush_l2=True, dry_run=False, batch=1, dtype=BF16, stream=None):
        """Measured plan search (mafat_search_measured): returns (candidates, best index), each
        candidate a dict with n_groups, cut (None for one group), grids [(n, m), ...],
        intermediate_bytes, predicted_mib, executed_flops, us_per_run (None if not timed) and
        status."""
        opt = SearchOptions()
        opt.struct_size = ctypes.sizeof(SearchOptions)
        opt.batch, opt.dtype, opt.include_one_group = batch, dtype, int(include_one_group)
        cut_arr = (i32 * max(1, len(cuts)))(*cuts)
        opt.n_cuts, opt.cuts = len(cuts), ctypes.cast(cut_arr, ctypes.POINTER(i32))
        opt.max_grid, opt.square_only, opt.budget_bytes = max_grid, int(square_only), budget_bytes
        opt.runs, opt.flush_l2, opt.dry_run = runs, int(flush_l2), int(dry_run)
        cap = 4096
        out = (SearchCandidate * cap)()
        n, best = i32(), i32()
        _check(lib.mafat_search_measured(self.handle, ctypes.byref(opt), _stream(stream), out, cap,
                                         ctypes.byref(n), ctypes.byref(best)))
        res = []
        for c in out[:min(n.value, cap)]:
            g = c.n_groups
            res.append({"n_groups": g, "cut": c.cut if g == 2 else None,
                        "grids": [(c.grid_n[i], c.grid_m[i]) for i in range(g)],
                        "intermediate_bytes": c.intermediate_bytes, "predicted_mib": c.predicted_mib,
                        "executed_flops": c.executed_flops,
                        "us_per_run": c.us_per_run if c.us_per_run >= 0 else None, "status": c.status})
        return res, best.value

    def close(self):
        if getattr(self, "handle", None):
            lib.mafat_net_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Plan:
    """mafat_plan_ex / mafat_run: fused-tile execution of a network on the current CUDA device."""

    def __init__(self, net, cut=None, grids=((1, 1),), batch=1, dtype=BF16, ring_slots=0, wave_tiles=0,
                 max_ctas=0, wait_timeout_ns=0, test_unpublished_task=-1, dry_run=False, trace=False,
                 force_nblk=0, force_mb=0, lookahead_items=0, tile_bounds=None, halo_reuse=False,
                 frame_major=False, chain=False, rect_blocks=False):
        self.net = net
        # cut: None (one group), the first layer of group 2, or a list of increasing cuts
        cut_list = [] if cut is None else (list(cut) if isinstance(cut, (list, tuple)) else [cut])
        n_groups = 1 + len(cut_list)
        grids = list(grids)[:n_groups]
        width = max(2, n_groups)
        gn = (i32 * width)(*[g[0] for g in grids] + [1] * (width - len(grids)))
        gm = (i32 * width)(*[g[1] for g in grids] + [1] * (width - len(grids)))
        cuts = (i32 * max(1, len(cut_list)))(*(cut_list or [0]))
        opt = PlanOptions()
        opt.struct_size = ctypes.sizeof(PlanOptions)
        opt.ring_slots, opt.wave_tiles, opt.max_ctas = ring_slots, wave_tiles, max_ctas
        opt.wait_timeout_ns = wait_timeout_ns
        opt.test_unpublished_task = test_unpublished_task
        opt.dry_run = 1 if dry_run else 0
        opt.trace = 1 if trace else 0
        opt.force_nblk, opt.force_mb = force_nblk, force_mb
        opt.lookahead_items = lookahead_items
        opt.halo_reuse = int(halo_reuse)
        opt.frame_major = int(frame_major)
        opt.chain = int(chain)
        opt.rect_blocks = int(rect_blocks)
        if tile_bounds is not None:
            # per group (rows, cols): the non-uniform tiling; kept alive with the plan
            flat = [v for rows, cols in list(tile_bounds)[:n_groups] for v in list(rows) + list(cols)]
            self._bounds = (i32 * len(flat))(*flat)
            opt.tile_bounds = ctypes.cast(self._bounds, ctypes.POINTER(i32))
        h = vp()
        _check(lib.mafat_plan_ex(net.handle, n_groups, cuts, gn, gm, batch, dtype, ctypes.byref(opt),
                                 ctypes.byref(h)))
        self.handle = h
        self.cut, self.grids, self.batch, self.dtype = cut, grids, batch, dtype

    def run(self, inp, out, stream=None):
        """mafat_run: inp NHWC [B][H][W][C] and out NHWC [B][H_out][W_out][C_out], both
        device tensors of the plan's dtype."""
        _check(lib.mafat_run(self.handle, _ptr(inp), _ptr(out), _stream(stream, inp)))

    def run_debug(self, inp, cut_out, out, stream=None):
        _check(lib.mafat_run_debug(self.handle, _ptr(inp), _ptr(cut_out), _ptr(out), _stream(stream, inp)))

    def run_noalloc(self, inp, out, stream=None):
        """Run an FP32 plan with its per-run scratch in the library's fixed 32 MiB
        device area (mafat_run_fp32_noalloc): no allocation at all, for callers
        that may not allocate device memory while they run.  Calls share the
        area and must not overlap on the GPU."""
        _check(lib.mafat_run_fp32_noalloc(self.handle, _ptr(inp), _ptr(out), _stream(stream, inp)))

    @staticmethod
    def noalloc_sync_status(stream=None, like=None):
        """Raises MafatError (ETIMEOUT / EDEVICE) if a device-side wait of an earlier
        run_noalloc call on the current device ran out (mafat_noalloc_sync_status)."""
        _check(lib.mafat_noalloc_sync_status(_stream(stream, like)))

    def run_host(self, inp_host, out_host, stream=None):
        """End to end on host tensors: inp_host NHWC [B][H][W][C] (the image batch as it
        comes, pinned for asynchronous copies), out_host NHWC; synchronises the stream."""
        _check(lib.mafat_run_host(self.handle, _ptr(inp_host), _ptr(out_host), _stream(stream)))

    def run_host_async(self, inp_host, out_host, stream=None):
        """Enqueue one frame on host tensors (two frames in flight); inp_host must stay
        unchanged and out_host unread until run_host_wait returns."""
        _check(lib.mafat_run_host_async(self.handle, _ptr(inp_host), _ptr(out_host), _stream(stream)))

    def run_host_wait(self):
        """Wait for every enqueued frame's output to reach host memory; raises on device errors."""
        _check(lib.mafat_run_host_wait(self.handle))

    def sync_status(self, stream=None, like=None):
        """Raises MafatError (ETIMEOUT / EDEVICE) if a device-side wait ran out."""
        _check(lib.mafat_sync_status(self.handle, _stream(stream, like)))

    def status(self, stream=None, like=None):
        return lib.mafat_sync_status(self.handle, _stream(stream, like))

    def tile_region(self, group, i, j, layer):
        a, b = _rect(), _rect()
        _check(lib.mafat_tile_region(self.handle, group, i, j, layer, a, b))
        return tuple(b), tuple(a)  # (out_rect, in_rect)

    def stats(self):
        s = PlanStats()
        s.struct_size = ctypes.sizeof(PlanStats)
        _check(lib.mafat_plan_stats(self.handle, ctypes.byref(s)))
        return {k: getattr(s, k) for k, _ in PlanStats._fields_ if k not in ("struct_size", "reserved")}

    def trace(self, stream=None):
        """Per-item records of the last run (plan made with trace=True): numpy uint64
        [n_items][10] = ticket taken, deps satisfied, accumulator ready, published (ns), SM,
        task << 16 | layer, first halo landed, last MMA issued (ns), ns waited for later
        halos, ns waited for streamed weight pieces."""
        import numpy as np
        n = self.stats()["n_items"]
        out = np.zeros((n, 10), dtype=np.uint64)
        _check(lib.mafat_plan_trace(self.handle, out.ctypes.data, out.size, _stream(stream)))
        return out

    def launches_per_run(self):
        return lib.mafat_launches_per_run(self.handle)

    def close(self):
        if getattr(self, "handle", None):
            lib.mafat_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def diag_umma(a_dev, b_dev, d_dev, n, a_in_tmem=False, stream=None):
    """One 128 x n x 16 bf16 tensor-core product d = a * b^T with the fused kernel's
    operand and accumulator layouts, A from shared or from tensor memory (mafat_diag_umma)."""
    _check(lib.mafat_diag_umma(_ptr(a_dev), _ptr(b_dev), _ptr(d_dev), n, int(a_in_tmem), _stream(stream, a_dev)))


def version():
    return lib.mafat_version().decode()


def from_planar(xp, C):
    """Host layout helper for the cut tensor of run_debug: octet-planar
    [B][C8][H][W][8] -> NHWC [B][H][W][C] (numpy)."""
    import numpy as np
    B, c8, H, W, _ = xp.shape
    return np.ascontiguousarray(xp.transpose(0, 2, 3, 1, 4).reshape(B, H, W, c8 * 8)[..., :C])
