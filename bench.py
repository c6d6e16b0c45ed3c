"""Throughput of fused-tile execution of the YOLOv2 first-16-layer front-end on GB300.

One step = one mafat_run of the whole plan (every fused layer group, every
tile) over one batch of synthetic input already resident in HBM.  Default
workload: 608x608x3, batch 1, bf16, two layer groups cut after layer 7, group 1
tiled 5x5 and group 2 tiled 2x2.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mafat|reference] [--workload NAME]

--impl reference times the CPU oracle (its plain fp32 build) on the host cores (the
only other place this script runs oracle code, together with the cpu_baseline leg).
Under torchrun (N > 1) every rank runs an independent replica on its own GPU
(the method does not shard a frame across devices); rank 0 reports the frames
of all ranks over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "frames/s (YOLOv2 first 16 layers, 608x608, bf16, fused tiles)"


def metric_of(name):
    """The metric line of a workload (the headline one for the default workload)."""
    wl = synth.WORKLOADS[name]
    if name == DEFAULT_WORKLOAD:
        return METRIC
    net = "YOLOv2 first 16 layers" if wl["layers"] == synth.YOLO16 else "YOLOv2 trunk, %d layers" % len(wl["layers"])
    return "frames/s (%s, %dx%d, %s, fused tiles)" % (net, wl["h"], wl["w"], wl["dtype"])
DEFAULT_WORKLOAD = "yolo16_608_5x5_c8_2x2"
L2_FLUSH_BYTES = 256 << 20
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
KERNEL_SOURCES = ["kernel_tc.cu", "sched.cuh", "device_types.h", "planner.cpp"]


def kernel_source_hash():
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2107_06960_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            p = json.load(fh)
        return float(p["bf16_tflops"]), float(p["bf16_tflops_sustained"]), float(p["hbm_gbs"]), "measured"
    except Exception:
        return 1900.0, 1700.0, 6800.0, "fallback"


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def reduce_max(pg, values, device):
    """Max over ranks of each value (the slowest rank's times); the values themselves at N = 1."""
    if pg is None:
        return [float(v) for v in values]
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def aggregate(units_per_rank, seconds_per_rank):
    """Whole-job throughput of independent replicas: all units over the slowest rank's time."""
    return float(sum(units_per_rank)) / float(max(seconds_per_rank))


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,utilization.gpu")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.QUERY, "--format=csv,noheader,nounits",
                 "-lms", "10"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            # nvidia-smi takes a while to start: wait (bounded) for its first line so that
            # the samples cover the timed region rather than the time after it
            t0 = time.time()
            while not self.lines and time.time() - t0 < 5.0 and self.proc.poll() is None:
                time.sleep(0.01)
            self.n_before = len(self.lines)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, busy, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        # the samples taken after the timed region started (the first line predates it)
        for ln in self.lines[self.n_before:] or self.lines[-1:]:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            try:
                busy.append(len(f) > 9 and float(f[9]) >= 50.0)
            except ValueError:
                busy.append(False)
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1"):
                    reasons.add(n)
        loaded = [c for c, b in zip(sm, busy) if b]
        use = loaded or sm
        return {"sm_mhz": statistics.median(use) if use else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm), "samples_under_load": len(loaded),
                "span": "every timed leg (device, chained, steady-state, end-to-end); median over samples with "
                        "GPU utilisation >= 50 %"}


def _best_of(n, fn):
    best = None
    for _ in range(n):
        t0 = time.perf_counter()
        fn()
        el = time.perf_counter() - t0
        best = el if best is None else min(best, el)
    return best


def cpu_oracle_timings(wl_names=(DEFAULT_WORKLOAD, "yolo16_416_1x3x3"), best_of=3):
    """The oracle as it stands, in its plain fp32 build (the same loops as the fp64 parity
    oracle, single precision), on the host cores: for each workload, single-threaded and
    with every core (OpenMP over output rows), best of `best_of` wall-clock runs.  All-core
    runs time whole frames; single-threaded runs time a centre crop of 1/16 of the frame's
    pixels and scale by the crop's share of the frame's FLOPs (the work per pixel is the
    same everywhere but at the image border)."""
    import oracle
    cores = os.cpu_count() or 1
    rows = []
    for name in wl_names:
        w = synth.workload(name)
        layers, params, x = w["layers"], w["params"], w["input"][0]
        full = oracle.conv_flops(layers, oracle.layer_shapes(layers, w["h"], w["w"], 3))
        side = w["h"] // 4
        y0 = (w["h"] - side) // 2
        crop = x[y0:y0 + side, y0:y0 + side]
        frac = oracle.conv_flops(layers, oracle.layer_shapes(layers, side, side, 3)) / full
        for threads in (1, cores):
            oracle.set_num_threads(threads, "f32")
            if threads == 1:
                t = _best_of(best_of, lambda: oracle.forward(layers, params, crop, precision="f32")) / frac
                sample = "%dx%d centre crop (%.4f of a frame's FLOPs), scaled" % (side, side, frac)
            else:
                t = _best_of(best_of, lambda: oracle.forward(layers, params, x, precision="f32"))
                sample = "whole %dx%d frame" % (w["h"], w["w"])
            rows.append({"workload": name, "threads": threads, "s_per_frame": t, "frames_per_s": 1.0 / t,
                         "gflop_per_s": full / t / 1e9, "sample": sample})
    oracle.set_num_threads(cores, "f32")
    return rows, cores


def run_reference(args, wl):
    """--impl reference: the CPU oracle timed per step on a bounded sample of the workload."""
    import oracle
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    layers, params = wl["layers"], wl["params"]
    full = oracle.conv_flops(layers, oracle.layer_shapes(layers, wl["h"], wl["w"], 3))
    cores = os.cpu_count() or 1
    oracle.set_num_threads(cores, "f32")
    # size the per-step sample so the whole run stays within about two minutes
    t0 = time.perf_counter()
    oracle.forward(layers, params, wl["input"][0][:152, :152], precision="f32")
    t_small = time.perf_counter() - t0
    est_full = t_small * (wl["h"] * wl["w"]) / (152 * 152)
    steps = args.steps + args.warmup
    side = wl["h"]
    while side > 64 and est_full * (side * side) / (wl["h"] * wl["w"]) * steps > 120.0:
        side //= 2
    side = max(16, side - side % 16)
    x = wl["input"][0][:side, :side]
    frac = oracle.conv_flops(layers, oracle.layer_shapes(layers, side, side, 3)) / full
    for _ in range(args.warmup):
        oracle.forward(layers, params, x, precision="f32")
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.forward(layers, params, x, precision="f32")
    el = time.perf_counter() - t0
    value = frac * args.steps / el
    sample = "%dx%d crop per step (%.4f of a frame's FLOPs), unfused forward, the oracle's fp32 build" % (
        side, side, frac)
    line = {
        "impl": "reference", "metric": metric_of(args.workload), "value": value, "unit": "frames/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": args.workload, "input": "%dx%dx3" % (wl["h"], wl["w"]), "batch": wl["batch"]},
        "cpu_baseline": {"value": value, "unit": "frames/s", "cores": oracle.num_threads("f32"), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "frames/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_sweep(args):
    """Plans of the 608x608 network over cut points and per-group grids (the paper's
    configuration space, Sec. 4 and Table 1): device-timed frames/s with L2 flushed before
    every step, Algorithm 1's prediction, the plan's intermediate bytes (tile scratch ring
    plus cut tensor) and the halo recompute, one JSON line each."""
    import torch
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    torch.cuda.set_device(0)
    wl = synth.workload(DEFAULT_WORKLOAD)
    H, W = wl["h"], wl["w"]
    net = mf.Net(wl["layers"], H, W, 3)
    net.set_params(wl["params"])
    xin = torch.from_numpy(wl["input"]).to(torch.bfloat16).cuda()
    sh = net.shape(len(wl["layers"]) - 1)
    out = torch.empty((1, sh[3], sh[4], sh[5]), dtype=torch.bfloat16, device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device="cuda")
    configs = [(None, [(t, t)]) for t in synth.SWEEP_GRIDS]
    configs += [(cut, [(t1, t1), (t2, t2)]) for cut in synth.SWEEP_CUTS
                for t1 in synth.SWEEP_GRIDS for t2 in synth.SWEEP_GRIDS]
    steps = max(20, min(args.steps, 200))
    best = None
    for cut, grids in configs:
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        plan = mf.Plan(net, cut, grids, batch=1, dtype=mf.BF16)
        st = plan.stats()
        torch.cuda.synchronize()
        plan_bytes = free0 - torch.cuda.mem_get_info()[0]
        for _ in range(3):
            plan.run(xin, out)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for a, b in ev:
            flush.fill_(1)
            a.record()
            plan.run(xin, out)
            b.record()
        torch.cuda.synchronize()
        plan.sync_status(like=out)
        times = [a.elapsed_time(b) for a, b in ev]
        ms = statistics.fmean(times)
        cut_bytes = 0
        if cut is not None:
            c = net.shape(cut - 1)
            cut_bytes = (c[5] + 7) // 8 * 8 * c[3] * c[4] * 2
        line = {"sweep": True, "cut": cut, "grids": "/".join("%dx%d" % gd for gd in grids),
                "frames_per_s": 1e3 / ms, "ms_mean": ms, "ms_median": statistics.median(times), "steps": steps,
                "predicted_mib_alg1": st["predicted_mib"],
                "intermediate_mb": (st["scratch_bytes"] + cut_bytes) / 1e6,
                "plan_device_mb": plan_bytes / 1e6,
                "executed_gflop": st["executed_flops"] / 1e9,
                "halo_recompute": st["executed_flops"] / st["useful_flops"] - 1.0, "work_items": st["n_items"]}
        print(json.dumps(line), flush=True)
        if best is None or ms < best["ms_mean"]:
            best = line
        plan.close()
    print(json.dumps({"sweep_best": best}), flush=True)
    # the same space through the library's measured search: candidates whose intermediates
    # exceed the L2 are refused, the rest timed on the device
    cands, bi = net.search_measured(cuts=synth.SWEEP_CUTS, max_grid=max(synth.SWEEP_GRIDS), runs=steps)
    timed = [c for c in cands if c["us_per_run"] is not None]
    print(json.dumps({"search_measured": {
        "candidates": len(cands), "timed": len(timed), "refused_over_l2": sum(c["status"] == mf.ENOFIT for c in cands),
        "best": cands[bi] if bi >= 0 else None,
        "benchmark_plan": next((c for c in cands if c["cut"] == 8 and c["grids"] == [(5, 5), (2, 2)]), None)}}),
        flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="mafat", choices=["mafat", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--frames-in-flight", type=int, default=16,
                    help="frames of the steady-state leg (one launch of a plan of this many frames, "
                         "frame f's second group overlapped with frame f+1's first); 0: skip it")
    ap.add_argument("--sweep", action="store_true",
                    help="time every plan of the 608x608 net over cuts {none, 2, 4, 8, 12} x grids 1..5 per "
                         "group (one JSON line per plan, then the fastest), instead of the benchmark line")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    wl = synth.workload(args.workload)

    if args.impl == "reference":
        run_reference(args, wl)
        return
    if args.sweep:
        run_sweep(args)
        return

    import torch
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf

    ws, rank, local = dist_env()
    pg = None
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        pg = dist
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    B, H, W = wl["batch"], wl["h"], wl["w"]
    net = mf.Net(wl["layers"], H, W, 3)
    net.set_params(wl["params"])
    dt = mf.BF16 if wl["dtype"] == "bf16" else mf.FP32
    tdt = torch.bfloat16 if dt == mf.BF16 else torch.float32
    plan = mf.Plan(net, wl["cut"], wl["grids"], batch=B, dtype=dt)
    st = plan.stats()
    sh = net.shape(len(wl["layers"]) - 1)
    xin = torch.from_numpy(wl["input"]).to(tdt).to(dev)  # NHWC [B][H][W][3], as the image comes
    out = torch.empty((B, sh[3], sh[4], sh[5]), dtype=tdt, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    for _ in range(args.warmup):
        plan.run(xin, out, stream=stream)
    plan.sync_status(stream=stream)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    for i in range(args.steps):
        flush.fill_(i)                       # write 256 MiB: evicts the 129 MB L2 (not timed)
        starts[i].record(stream)
        plan.run(xin, out, stream=stream)    # one kernel launch
        ends[i].record(stream)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    plan.sync_status(stream=stream)
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    dev_s = sum(step_ms) / 1e3

    # The same 1-frame plan with on-chip chaining of the 3x3 -> 1x1 pairs that fit one TMEM
    # buffer (plan option chain=1): its device time, measured the same way, and its task count.
    chained = None
    if B == 1 and dt == mf.BF16:
        plan_c = mf.Plan(net, wl["cut"], wl["grids"], batch=B, dtype=dt, chain=True)
        st_c = plan_c.stats()
        if st_c["n_tasks"] < st["n_tasks"]:
            for _ in range(args.warmup):
                plan_c.run(xin, out, stream=stream)
            c_steps = max(20, min(args.steps // 4, 500))
            c_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(c_steps)]
            torch.cuda.synchronize()
            for a, b in c_ev:
                flush.fill_(1)
                a.record(stream)
                plan_c.run(xin, out, stream=stream)
                b.record(stream)
            torch.cuda.synchronize()
            plan_c.sync_status(stream=stream)
            c_ms = statistics.fmean(a.elapsed_time(b) for a, b in c_ev)
            chained = {"ms_per_frame": c_ms, "value": 1e3 / c_ms, "unit": "frames/s", "steps": c_steps,
                       "n_tasks": st_c["n_tasks"], "n_tasks_unchained": st["n_tasks"],
                       "mode": "plan option chain=1: a 3x3 and the 1x1 after it in one item, the intermediate "
                               "kept in TMEM; same L2 flush per step"}
        plan_c.close()

    # Steady state with frames in flight: one launch of a K-frame plan, whose hand-out order
    # overlaps frame f's second group (a chain of small-map stages that leaves SMs idle)
    # with frame f + 1's first.  Each frame is still a 608x608 batch-1 image; the L2 is
    # flushed before every launch as in the device leg.
    ss = None
    K = args.frames_in_flight
    if K > 1 and B == 1 and wl["cut"] is not None:
        plan_k = mf.Plan(net, wl["cut"], wl["grids"], batch=K, dtype=dt)
        st_k = plan_k.stats()
        xk = torch.from_numpy(synth.make_input(K, H, W, 3, synth.SEED_BASE + 77, wl["dtype"]))
        xk = xk.to(tdt).to(dev)
        outk = torch.empty((K, sh[3], sh[4], sh[5]), dtype=tdt, device=dev)
        for _ in range(args.warmup):
            plan_k.run(xk, outk, stream=stream)
        plan_k.sync_status(stream=stream)
        ss_steps = max(3, min(args.steps // 20, 100))
        s_ev = [torch.cuda.Event(enable_timing=True) for _ in range(ss_steps)]
        e_ev = [torch.cuda.Event(enable_timing=True) for _ in range(ss_steps)]
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        for i in range(ss_steps):
            flush.fill_(i)
            s_ev[i].record(stream)
            plan_k.run(xk, outk, stream=stream)
            e_ev[i].record(stream)
        torch.cuda.synchronize()
        plan_k.sync_status(stream=stream)
        ss_ms = [a.elapsed_time(b) for a, b in zip(s_ev, e_ev)]
        # self-check outside the timed region: the first and last frames of the K-frame
        # launch against the same frames run one at a time through the 1-frame plan
        one = torch.empty_like(out)
        ss_err = 0.0
        for f in (0, K - 1):
            plan.run(xk[f:f + 1], one, stream=stream)
            plan.sync_status(stream=stream)
            ref = one.float()
            ss_err = max(ss_err, float((outk[f:f + 1].float() - ref).abs().max()) / max(float(ref.abs().max()), 1e-30))
        ss = {"frames_in_flight": K, "launches": ss_steps, "seconds": sum(ss_ms) / 1e3,
              "overlapped": bool(st_k["frames_overlapped"]), "items": st_k["n_items"], "check": ss_err}
        plan_k.close()
        del xk, outk, one

    # End to end through the C ABI on pinned host buffers, every step's upload of its
    # input and read-back of its output inside the timed region.  Streamed the way a
    # serving loop would (mafat_run_host_async: the upload of one frame overlaps the run
    # of the previous one); the synchronous call's rate is reported beside it.
    xh = torch.from_numpy(wl["input"]).to(tdt).pin_memory()   # NHWC image batch as it comes
    ohs = [torch.empty(out.shape, dtype=tdt).pin_memory() for _ in range(2)]
    oh = ohs[0]
    for i in range(4):
        plan.run_host_async(xh, ohs[i % 2], stream=stream)
    plan.run_host_wait()
    e2e_steps = max(5, min(args.steps, 200))
    t0 = time.perf_counter()
    for i in range(e2e_steps):
        plan.run_host_async(xh, ohs[i % 2], stream=stream)
    plan.run_host_wait()
    e2e_s = time.perf_counter() - t0
    for _ in range(2):
        plan.run_host(xh, oh, stream=stream)
    sync_steps = max(5, min(args.steps, 50))
    t0 = time.perf_counter()
    for _ in range(sync_steps):
        plan.run_host(xh, oh, stream=stream)
    sync_s = time.perf_counter() - t0
    # the sampler ran through every timed leg (device, chained, steady-state, end-to-end)
    clk = clocks.stop()

    dev_s_max, e2e_s_max, sync_s_max, ss_s_max = reduce_max(
        pg, [dev_s, e2e_s, sync_s, ss["seconds"] if ss else 0.0], dev)
    if rank != 0:
        if pg:
            pg.destroy_process_group()
        return

    frames = B * args.steps
    value = aggregate([frames] * ws, [dev_s_max])
    e2e_value = aggregate([B * e2e_steps] * ws, [e2e_s_max])
    peak_burst, peak_sus, hbm, peak_src = measured_peaks()
    avg_launch_s = dev_s / args.steps
    achieved_tf = st["useful_flops"] / avg_launch_s / 1e12
    traffic = None
    ss_traffic = None
    try:
        with open(TRAFFIC_FILE) as fh:
            tr = json.load(fh)
        h = kernel_source_hash()
        ent = tr.get(args.workload)
        if ent and ent.get("kernel_source_hash") == h:
            traffic = ent["dram_bytes_per_launch"]
        if ss is not None:
            ent = tr.get("%s@%d" % (args.workload, ss["frames_in_flight"]))
            if ent and ent.get("kernel_source_hash") == h:
                ss_traffic = ent["dram_bytes_per_launch"] / ss["frames_in_flight"]
    except Exception:
        pass

    cpu = None
    if not args.no_cpu_baseline:
        names = [args.workload] + (["yolo16_416_1x3x3"] if args.workload == DEFAULT_WORKLOAD else [])
        rows, cores = cpu_oracle_timings(names)
        head = next(r for r in rows if r["workload"] == args.workload and r["threads"] == cores)
        cpu = {"value": head["frames_per_s"], "unit": "frames/s", "cores": cores, "kind": "oracle",
               "precision": "f32 (the oracle's loops built in single precision; parity uses its fp64 build)",
               "sample": "%s, all %d host cores, best of 3" % (head["sample"], cores),
               "timings": rows}

    line = {
        "metric": metric_of(args.workload), "value": value, "unit": "frames/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dev_s_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if dt == mf.BF16 else "f32", "data": "synthetic",
        "config": {
            "workload": args.workload, "input": "%dx%dx3" % (H, W), "batch": B,
            "cut": wl["cut"], "grids": "/".join("%dx%d" % tuple(gd) for gd in wl["grids"]),
            "l2": "flushed before every timed step (256 MiB write, not timed)",
            "e2e_l2": "not flushed between streamed frames (a serving loop keeps the %.1f MB of weights in L2)"
                      % (st["weight_bytes"] / 1e6),
            "useful_gflop_per_frame": st["useful_flops"] / B / 1e9,
            "executed_gflop_per_frame": st["executed_flops"] / B / 1e9,
            "halo_recompute": st["executed_flops"] / st["useful_flops"] - 1.0,
            "issued_gflop_per_frame": st["issued_flops"] / B / 1e9,
            "group_io_mb_per_frame": st["group_io_bytes"] / B / 1e6,
            "weight_mb": st["weight_bytes"] / 1e6,
            "predicted_mib_alg1": st["predicted_mib"],
            "ctas": st["max_ctas"], "work_items": st["n_items"],
            "step_ms_min": min(step_ms), "step_ms_median": statistics.median(step_ms),
        },
        "roofline": {"bound": "tensor", "achieved": achieved_tf, "peak": peak_burst, "unit": "TFLOP/s",
                     "frac": achieved_tf / peak_burst, "traffic": traffic,
                     "kernel": "mafat_tc_kernel", "flops": "useful (unfused network) per launch",
                     "peak_source": "%s dense bf16 burst" % peak_src},
        "e2e": {"value": e2e_value, "unit": "frames/s", "h2d_bytes_per_step": int(xh.numel() * xh.element_size()),
                "d2h_bytes_per_step": int(oh.numel() * oh.element_size()),
                "mode": "mafat_run_host_async, two frames in flight, copies in the timed region",
                "sync_call_value": aggregate([B * sync_steps] * ws, [sync_s_max])},
        "gpu_launches": args.steps * plan.launches_per_run(),
        "clocks": clk,
    }
    if ss is not None:
        ss_value = aggregate([ss["frames_in_flight"] * ss["launches"]] * ws, [ss_s_max])
        ss_tf = st["useful_flops"] / B * ss_value / ws / 1e12
        line["steady_state"] = {
            "value": ss_value, "unit": "frames/s", "frames_in_flight": ss["frames_in_flight"],
            "ms_per_frame": 1e3 * ss_s_max / (ss["frames_in_flight"] * ss["launches"]),
            "launches": ss["launches"], "gpu_launches": ss["launches"] * plan.launches_per_run(),
            "work_items_per_launch": ss["items"], "frames_overlapped": ss["overlapped"],
            "check_vs_one_frame": {"max_rel_err": ss["check"], "frames": [0, ss["frames_in_flight"] - 1],
                                   "tolerance": 2e-2},
            "roofline_frac": ss_tf / peak_burst, "achieved_tflops": ss_tf, "dram_bytes_per_frame": ss_traffic,
            "mode": "one launch of a %d-frame plan per step (frame f's second group overlapped with frame "
                    "f+1's first), L2 flushed before every launch" % ss["frames_in_flight"]}
    if chained is not None:
        line["chained"] = chained
    if cpu is not None:
        line["cpu_baseline"] = cpu
    print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
