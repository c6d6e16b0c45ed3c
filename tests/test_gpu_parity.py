"""Parity of the CUDA path (through the C ABI) with the fp64 oracle on the same seeded inputs.

Tolerances (per layer-group output, max |err| <= tol * max |ref|):
  * bf16 tensor-core path: 2e-2 (activations, weights and every layer output in bf16);
  * fp32 check path: 1e-4.
Single-layer cases are held to a per-element bound of bf16 rounding instead.
Every fused-tile plan of a network must give bit-identical results (the
tiling changes only which tile computes a pixel, never how).
"""
import numpy as np
import pytest

import oracle
import synth
from tests.gpu_util import rel_err, run_plan

pytestmark = pytest.mark.gpu

TOL_BF16 = 2e-2
TOL_FP32 = 1e-4


@pytest.fixture(scope="module")
def mf():
    import torch
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    # The kernels read shared memory through descriptors whose field assignment
    # the diagnostic product confirms; never launch them if it does not hold.
    rng = np.random.default_rng(0)
    a = torch.from_numpy(rng.standard_normal((128, 16)).astype(np.float32)).to(torch.bfloat16).cuda()
    b = torch.from_numpy(rng.standard_normal((256, 16)).astype(np.float32)).to(torch.bfloat16).cuda()
    d = torch.zeros((128, 256), dtype=torch.float32, device="cuda")
    mf.diag_umma(a, b, d, 256)
    ref = a.double().cpu().numpy() @ b.double().cpu().numpy().T
    if not np.allclose(d.cpu().numpy(), ref, rtol=1e-5, atol=1e-5):
        pytest.fail("tensor-core descriptor layout check failed; not launching the fused kernels")
    return mf


_REF = {}


def _oracle_groups(layers, params, x, cut, key=None):
    """Oracle group outputs of every frame (cached by key)."""
    if key is not None and key in _REF:
        return _REF[key]
    res = [oracle.group_outputs(layers, params, x[b], cut) for b in range(x.shape[0])]
    if key is not None:
        _REF[key] = res
    return res


def _check_groups(got_cut, got_out, refs, cut, tol, frames=None):
    frames = range(len(refs)) if frames is None else frames
    for b in frames:
        if cut is not None:
            e = rel_err(got_cut[b], refs[b][0])
            assert e <= tol, "frame %d cut tensor: rel err %.3g > %.3g" % (b, e, tol)
        e = rel_err(got_out[b], refs[b][-1])
        assert e <= tol, "frame %d output: rel err %.3g > %.3g" % (b, e, tol)


# ---------------------------------------------------------------------------
# fp32 check path
# ---------------------------------------------------------------------------

def test_fp32_tiny3_64_grid2x2(mf):
    wl = synth.workload("tiny3_64_fp32")
    _, out = run_plan(mf, wl["layers"], wl["params"], wl["input"], None, wl["grids"], mf.FP32)
    refs = _oracle_groups(wl["layers"], wl["params"], wl["input"], None)
    _check_groups(None, out, refs, None, TOL_FP32)


@pytest.mark.parametrize("cut,grids", [(None, [(1, 1)]), (None, [(3, 2)]), (2, [(5, 5), (2, 2)]),
                                       (4, [(3, 3), (4, 4)]), (8, [(5, 5), (2, 2)]), (12, [(5, 5), (5, 5)])])
def test_fp32_yolo16_96(mf, cut, grids):
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 31, "fp32")
    x = synth.make_input(2, 96, 96, 3, 32, "fp32")
    c, out = run_plan(mf, layers, params, x, cut, grids, mf.FP32)
    refs = _oracle_groups(layers, params, x, cut, ("fp32_96", cut is None and 16 or cut))
    _check_groups(c, out, refs, cut, TOL_FP32)


@pytest.mark.parametrize("name", ["yolo16_416_1x3x3", "yolo16_608_5x5_c8_2x2"])
def test_fp32_full_size(mf, name):
    wl = synth.WORKLOADS[name]
    params = synth.make_params(wl["layers"], 3, wl["seed"], "fp32")
    x = synth.make_input(1, wl["h"], wl["w"], 3, wl["seed"], "fp32")
    c, out = run_plan(mf, wl["layers"], params, x, wl["cut"], wl["grids"], mf.FP32)
    refs = _oracle_groups(wl["layers"], params, x, wl["cut"])
    _check_groups(c, out, refs, wl["cut"], TOL_FP32)


# ---------------------------------------------------------------------------
# bf16 tensor-core path: single layers at a per-element bound
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("cin,cout,k,pool,h,w,grid", [
    (3, 32, 3, True, 36, 28, (2, 3)),     # first layer: 8 padded channels, tap-paired K steps, fused pool
    (3, 8, 3, False, 19, 23, (1, 1)),     # output channels padded to the MMA N of 16
    (32, 64, 3, True, 40, 24, (3, 2)),    # one 32-channel chunk
    (64, 128, 3, False, 37, 29, (2, 2)),  # ragged blocks in both directions
    (128, 64, 1, False, 21, 30, (2, 1)),  # 1x1, two 64-channel chunks
    (256, 512, 3, False, 20, 18, (1, 2)), # two output-channel blocks, four chunks
    (512, 256, 1, False, 19, 19, (2, 2)),
    (16, 16, 3, True, 18, 34, (4, 4)),    # smallest K chunk (2 octets)
    (3, 32, 3, True, 36, 40, (2, 3)),     # RGB rows of 240 bytes: raw rows widened to 8 channels in the kernel
    (3, 16, 3, False, 18, 56, (1, 8)),    # RGB, tiles starting at every column mod 8: all raw-row alignments
    (4, 16, 3, False, 21, 34, (3, 2)),    # 4 channels, rows of 272 bytes, ragged blocks
    (1, 16, 3, True, 20, 24, (2, 2)),     # 1 channel
    (7, 16, 3, False, 17, 16, (1, 1)),    # 7 channels
    (8, 32, 3, True, 20, 22, (2, 2)),     # 8 channels: the NHWC input is one octet plane
    (32, 24, 3, True, 34, 30, (2, 2)),    # pooled 32-column unit with its last octet past cout
    (64, 40, 3, True, 26, 42, (1, 2)),    # pooled, N = 48: 16-column units
    (64, 96, 1, True, 32, 16, (2, 1)),    # pooled 1x1, three 32-column units per block
])
def test_bf16_single_layer(mf, cin, cout, k, pool, h, w, grid):
    layers = [("conv", k, 1, (k - 1) // 2, cout)] + ([("max", 2, 2, 0, 0)] if pool else [])
    params = synth.make_params(layers, cin, 1000 + cin + cout + k, "bf16")
    x = synth.make_input(1, h, w, cin, 2000 + cin, "bf16")
    _, out = run_plan(mf, layers, params, x, None, [grid], mf.BF16)
    ref = _oracle_groups(layers, params, x, None)[0][-1]
    got = out[0]
    assert np.isfinite(got).all()
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -12 * np.abs(ref).max()
    bad = np.abs(got - ref) > bound
    assert not bad.any(), "%d of %d elements out of bound; worst %.3g" % (
        bad.sum(), bad.size, float(np.abs(got - ref).max()))


def _issued(mf, layers, h, w, c, cut, grids, dtype, **kw):
    net = mf.Net(layers, h, w, c)
    net.set_params(synth.make_params(layers, c, 1, "fp32"))
    return mf.Plan(net, cut, grids, dtype=dtype, dry_run=True, **kw).stats()["issued_flops"]


@pytest.mark.parametrize("cin,cout,k,h,w,grid,mb", [
    (64, 64, 3, 40, 14, (1, 1), 0),     # pitch 16: 5 runs of 128 pixels instead of 6 rectangles
    (256, 512, 3, 38, 38, (2, 2), 0),   # the benchmark's 38x38 3x3 layers: 19x19 regions, pitch 24
    (512, 256, 1, 38, 38, (2, 2), 0),   # and its 1x1 layers, pitch 24
    (128, 64, 1, 33, 31, (1, 1), 0),    # pitch 32, a ragged last run
    (32, 48, 3, 70, 30, (1, 1), 0),     # pitch 32, output channels padded to the MMA N
    (32, 48, 3, 70, 30, (1, 1), 4),     # four runs per item (one accumulator each)
    (64, 32, 3, 99, 14, (3, 1), 2),     # two runs per item, 5 runs per task (3 + 2)
])
def test_bf16_flat_blocks_match_rectangles_and_oracle(mf, cin, cout, k, h, w, grid, mb):
    # A convolution without a pool whose regions are narrow reads them as flattened rows
    # (rect_blocks=False, the default); 16x8 rectangles (rect_blocks=True) compute every
    # pixel with the same products in the same order, so the outputs are bit-identical.
    layers = [("conv", k, 1, (k - 1) // 2, cout)]
    kw = dict(force_mb=mb) if mb else {}
    assert (_issued(mf, layers, h, w, cin, None, [grid], mf.BF16, **kw) <
            _issued(mf, layers, h, w, cin, None, [grid], mf.BF16, rect_blocks=True, **kw)), "no flat stage"
    params = synth.make_params(layers, cin, 3000 + cin + cout + k, "bf16")
    x = synth.make_input(1, h, w, cin, 4000 + cin, "bf16")
    _, flat = run_plan(mf, layers, params, x, None, [grid], mf.BF16, plan_kwargs=kw)
    _, rect = run_plan(mf, layers, params, x, None, [grid], mf.BF16, plan_kwargs=dict(rect_blocks=True, **kw))
    assert np.array_equal(flat, rect)
    ref = _oracle_groups(layers, params, x, None)[0][-1]
    bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -12 * np.abs(ref).max()
    bad = np.abs(flat[0] - ref) > bound
    assert not bad.any(), "%d of %d elements out of bound; worst %.3g" % (
        bad.sum(), bad.size, float(np.abs(flat[0] - ref).max()))


def test_bf16_flat_blocks_random_shapes(mf):
    # seeded random single convolutions (1x1 and 3x3, channel counts, map sizes, grids and
    # forced blocks per item) among those that the planner runs in flat blocks: bit-identical
    # to 16x8 rectangles and within the per-element bf16 bound of the oracle
    rng = np.random.default_rng(2107)
    done = 0
    for _ in range(2000):
        if done == 10:
            break
        cin = int(rng.choice([16, 32, 64, 128]))
        cout = int(rng.choice([16, 48, 64, 96, 128]))
        k = int(rng.choice([1, 3]))
        h, w = int(rng.integers(8, 72)), int(rng.integers(5, 40))
        grid = [(1, 1), (2, 1), (1, 2), (2, 2), (3, 2)][int(rng.integers(0, 5))]
        mb = int(rng.choice([0, 0, 2, 4]))
        layers = [("conv", k, 1, (k - 1) // 2, cout)]
        kw = dict(force_mb=mb) if mb else {}
        try:
            flat_work = _issued(mf, layers, h, w, cin, None, [grid], mf.BF16, **kw)
            rect_work = _issued(mf, layers, h, w, cin, None, [grid], mf.BF16, rect_blocks=True, **kw)
        except mf.MafatError:
            continue  # a shape the planner refuses (e.g. more blocks per item than fit)
        if flat_work >= rect_work:
            continue
        params = synth.make_params(layers, cin, 5000 + done, "bf16")
        x = synth.make_input(1, h, w, cin, 6000 + done, "bf16")
        _, flat = run_plan(mf, layers, params, x, None, [grid], mf.BF16, plan_kwargs=kw)
        _, rect = run_plan(mf, layers, params, x, None, [grid], mf.BF16, plan_kwargs=dict(rect_blocks=True, **kw))
        case = (cin, cout, k, h, w, grid, mb)
        assert np.array_equal(flat, rect), case
        ref = _oracle_groups(layers, params, x, None)[0][-1]
        bound = 2.0 ** -8 * np.abs(ref) + 2.0 ** -12 * np.abs(ref).max()
        assert not (np.abs(flat[0] - ref) > bound).any(), case
        done += 1
    assert done == 10


def test_fp32_flat_blocks_match_rectangles_and_oracle(mf):
    # a 3x3, a 1x1 and a 3x3 on 2x2 tiles of 38x38: 20, 20 and 19-pixel regions run
    # flattened (pitch 24), the later ones from the tile buffers of the scratch ring, in the
    # fp32 check kernel as in the bf16 one
    layers = [("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 32), ("conv", 3, 1, 1, 32)]
    assert (_issued(mf, layers, 38, 38, 16, None, [(2, 2)], mf.FP32) <
            _issued(mf, layers, 38, 38, 16, None, [(2, 2)], mf.FP32, rect_blocks=True))
    params = synth.make_params(layers, 16, 71, "fp32")
    x = synth.make_input(2, 38, 38, 16, 72, "fp32")
    _, flat = run_plan(mf, layers, params, x, None, [(2, 2)], mf.FP32)
    _, rect = run_plan(mf, layers, params, x, None, [(2, 2)], mf.FP32, plan_kwargs=dict(rect_blocks=True))
    assert np.array_equal(flat, rect)
    _check_groups(None, flat, _oracle_groups(layers, params, x, None), None, TOL_FP32)
    pb = synth.make_params(layers, 16, 73, "bf16")
    xb = synth.make_input(2, 38, 38, 16, 74, "bf16")
    _, fb = run_plan(mf, layers, pb, xb, None, [(2, 2)], mf.BF16)
    _, rb = run_plan(mf, layers, pb, xb, None, [(2, 2)], mf.BF16, plan_kwargs=dict(rect_blocks=True))
    assert np.array_equal(fb, rb)
    _check_groups(None, fb, _oracle_groups(layers, pb, xb, None), None, TOL_BF16)


def test_bf16_608_flat_matches_rectangles(mf):
    # the benchmark plan: layers 12-15 (19-20 pixel regions after the cut) run flattened
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    c1, o1 = run_plan(mf, wl["layers"], wl["params"], wl["input"], 8, wl["grids"], mf.BF16)
    c0, o0 = run_plan(mf, wl["layers"], wl["params"], wl["input"], 8, wl["grids"], mf.BF16,
                      plan_kwargs=dict(rect_blocks=True))
    assert np.array_equal(o1, o0) and np.array_equal(c1, c0)


# ---------------------------------------------------------------------------
# bf16 tensor-core path: whole YOLOv2 front-end
# ---------------------------------------------------------------------------

def test_bf16_tiny3_64_grid2x2(mf):
    layers = synth.TINY3
    params = synth.make_params(layers, 3, synth.SEED_BASE, "bf16")
    x = synth.make_input(1, 64, 64, 3, synth.SEED_BASE, "bf16")
    _, out = run_plan(mf, layers, params, x, None, [(2, 2)], mf.BF16)
    refs = _oracle_groups(layers, params, x, None)
    _check_groups(None, out, refs, None, TOL_BF16)


@pytest.mark.parametrize("cut,grids", [(None, [(1, 1)]), (None, [(3, 3)]), (2, [(5, 5), (2, 2)]),
                                       (4, [(4, 4), (3, 3)]), (8, [(5, 5), (2, 2)]), (8, [(1, 1), (1, 1)]),
                                       (12, [(5, 5), (5, 5)]), (12, [(7, 2), (1, 3)]),
                                       (8, [(2, 2), (5, 5)]), (4, [(3, 4), (4, 3)])])
def test_bf16_yolo16_96_batch2(mf, cut, grids):
    # two frames in one launch: with two groups the second frame's first group is handed
    # out between the first frame's second-group stages
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 41, "bf16")
    x = synth.make_input(2, 96, 96, 3, 42, "bf16")
    c, out = run_plan(mf, layers, params, x, cut, grids, mf.BF16)
    refs = _oracle_groups(layers, params, x, cut, ("bf16_96", cut is None and 16 or cut))
    _check_groups(c, out, refs, cut, TOL_BF16)


@pytest.mark.parametrize("cut,grids", [(8, [(3, 3), (2, 2)]), (4, [(2, 2), (2, 1)]), (None, [(2, 2)])])
def test_bf16_smallest_map_batch3(mf, cut, grids):
    # 32x32 input: the 16-layer net ends at 2x2, group 1 at cut 8 ends at 4x4, so tiles
    # shrink to one or two pixels; three frames in one launch
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, synth.SEED_BASE + 80, "bf16")
    x = synth.make_input(3, 32, 32, 3, synth.SEED_BASE + 80, "bf16")
    c, out = run_plan(mf, layers, params, x, cut, grids, mf.BF16)
    for f in range(3):
        refs = oracle.group_outputs(layers, params, x[f], cut)
        assert rel_err(out[f], refs[-1]) <= TOL_BF16
        if cut is not None:
            assert rel_err(c[f], refs[0]) <= TOL_BF16


@pytest.mark.parametrize("name", ["yolo16_416_1x3x3", "yolo16_608_5x5_c8_2x2"])
def test_bf16_full_size(mf, name):
    wl = synth.workload(name)
    c, out = run_plan(mf, wl["layers"], wl["params"], wl["input"], wl["cut"], wl["grids"], mf.BF16)
    refs = _oracle_groups(wl["layers"], wl["params"], wl["input"], wl["cut"], name)
    _check_groups(c, out, refs, wl["cut"], TOL_BF16)


@pytest.mark.parametrize("name", ["yolo25_96_2x2_c8_1x1", "yolo25_608_5x5_c8_2x2"])
def test_bf16_yolov2_trunk(mf, name):
    # a second workload: the whole YOLOv2 trunk, 1024-channel 3x3 layers (16 input chunks,
    # 1.2 MB of weights streamed per work item) after the fifth pooling
    wl = synth.workload(name)
    c, out = run_plan(mf, wl["layers"], wl["params"], wl["input"], wl["cut"], wl["grids"], mf.BF16)
    refs = _oracle_groups(wl["layers"], wl["params"], wl["input"], wl["cut"], name)
    _check_groups(c, out, refs, wl["cut"], TOL_BF16)


def test_fp32_yolov2_trunk_96(mf):
    layers = synth.YOLO25
    params = synth.make_params(layers, 3, 51, "fp32")
    x = synth.make_input(1, 96, 96, 3, 52, "fp32")
    c, out = run_plan(mf, layers, params, x, 8, [(2, 2), (1, 1)], mf.FP32)
    _check_groups(c, out, _oracle_groups(layers, params, x, 8), 8, TOL_FP32)


def test_bf16_608_frames_in_flight(mf):
    # three 608x608 frames in one launch, frame f's second group overlapped with frame
    # f + 1's first in the hand-out order: bit-identical to the frame-major order (same
    # items, only their order differs), every frame within the bf16 tolerance of the same
    # frame run alone (1x1 layers use other channel blocks there), the first frame
    # against the oracle
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, cut, grids = wl["layers"], wl["params"], wl["cut"], wl["grids"]
    x = np.concatenate([wl["input"], synth.make_input(2, 608, 608, 3, synth.SEED_BASE + 90, "bf16")], 0)
    c3, o3 = run_plan(mf, layers, params, x, cut, grids, mf.BF16)
    cm, om = run_plan(mf, layers, params, x, cut, grids, mf.BF16, plan_kwargs={"frame_major": True})
    assert np.array_equal(o3, om) and np.array_equal(c3, cm)
    for f in range(3):
        c1, o1 = run_plan(mf, layers, params, x[f:f + 1], cut, grids, mf.BF16)
        assert rel_err(o3[f], o1[0]) <= TOL_BF16 and rel_err(c3[f], c1[0]) <= TOL_BF16, "frame %d" % f
        assert np.array_equal(c3[f], c1[0]), "frame %d: the first group has the same items" % f
    refs = _oracle_groups(layers, params, wl["input"], cut, "yolo16_608_5x5_c8_2x2")
    _check_groups(c3[:1], o3[:1], refs, cut, TOL_BF16)


def test_bf16_1216_batch8_stress(mf):
    wl = synth.workload("yolo16_1216_b8_8x8_c8_4x4")
    c, out = run_plan(mf, wl["layers"], wl["params"], wl["input"], wl["cut"], wl["grids"], mf.BF16)
    assert np.isfinite(out).all() and np.isfinite(c).all()
    for b in (0, 7):   # two frames against the oracle (each is about 100 GFLOP of fp64)
        ref = oracle.group_outputs(wl["layers"], wl["params"], wl["input"][b], wl["cut"])
        assert rel_err(c[b], ref[0]) <= TOL_BF16
        assert rel_err(out[b], ref[1]) <= TOL_BF16


def test_bf16_608_plan_sweep_is_plan_independent(mf):
    # cut after layer 1, 3, 7, 11 x per-group grids 1..5 (100 plans).  With the MMA
    # shapes held fixed (32 output channels x one 16x8 block per item) every plan
    # must give bit-identical outputs -- tiling changes only which tile computes a
    # pixel, never how -- and equal the oracle within tolerance.
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, x = wl["layers"], wl["params"], wl["input"]
    refs = _oracle_groups(layers, params, x, 8, "yolo16_608_5x5_c8_2x2")
    base = None
    for cut in synth.SWEEP_CUTS:
        for t1 in synth.SWEEP_GRIDS:
            for t2 in synth.SWEEP_GRIDS:
                c, out = run_plan(mf, layers, params, x, cut, [(t1, t1), (t2, t2)], mf.BF16,
                                  plan_kwargs=dict(force_nblk=32, force_mb=1))
                if base is None:
                    base = out
                    assert rel_err(out[0], refs[0][-1]) <= TOL_BF16
                assert np.array_equal(out, base), "plan %d/%dx%d/%dx%d differs" % (cut, t1, t1, t2, t2)


def test_bf16_608_every_sweep_plan_default_shapes(mf):
    # every plan the benchmark's sweep times (one group with grids 1..5, and cut after
    # layer 1, 3, 7, 11 x per-group grids 1..5), with the MMA shapes the planner picks for
    # it: the cut tensor and the output within tolerance of one layer-by-layer oracle pass
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, x = wl["layers"], wl["params"], wl["input"]
    outs = oracle.forward(layers, params, x[0])
    plans = [(None, [(t, t)]) for t in synth.SWEEP_GRIDS]
    plans += [(cut, [(t1, t1), (t2, t2)]) for cut in synth.SWEEP_CUTS
              for t1 in synth.SWEEP_GRIDS for t2 in synth.SWEEP_GRIDS]
    for cut, grids in plans:
        c, out = run_plan(mf, layers, params, x, cut, grids, mf.BF16)
        e = rel_err(out[0], outs[-1])
        assert e <= TOL_BF16, "plan %s %s output: rel err %.3g" % (cut, grids, e)
        if cut is not None:
            e = rel_err(c[0], outs[cut - 1])
            assert e <= TOL_BF16, "plan %s %s cut tensor: rel err %.3g" % (cut, grids, e)


def test_bf16_608_nonuniform_tiling(mf):
    # non-uniform tile bounds: the output equals the oracle's, and with the MMA shapes held
    # fixed it is bit-identical to the even grid's
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, x = wl["layers"], wl["params"], wl["input"]
    bounds = [([0, 20, 30, 45, 60, 76], [0, 12, 30, 50, 64, 76]), ([0, 15, 38], [0, 24, 38])]
    outs = oracle.forward(layers, params, x[0])
    c, out = run_plan(mf, layers, params, x, 8, [(5, 5), (2, 2)], mf.BF16, plan_kwargs=dict(tile_bounds=bounds))
    assert rel_err(out[0], outs[-1]) <= TOL_BF16 and rel_err(c[0], outs[7]) <= TOL_BF16
    fixed = dict(force_nblk=32, force_mb=1)
    _, a = run_plan(mf, layers, params, x, 8, [(5, 5), (2, 2)], mf.BF16, plan_kwargs=dict(tile_bounds=bounds, **fixed))
    _, b = run_plan(mf, layers, params, x, 8, [(5, 5), (2, 2)], mf.BF16, plan_kwargs=fixed)
    assert np.array_equal(a, b)


@pytest.mark.parametrize("cut,grids", [(8, [(5, 5), (2, 2)]), (None, [(3, 3)]), (2, [(4, 4), (3, 3)]),
                                       (12, [(3, 2), (2, 3)])])
def test_bf16_yolo16_96_halo_reuse_batch2(mf, cut, grids):
    # inter-tile reuse (tiles read their neighbours' parts of the previous layer): the same
    # outputs as the oracle, and bit-identical to halo recompute with fixed MMA shapes
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 41, "bf16")
    x = synth.make_input(2, 96, 96, 3, 42, "bf16")
    c, out = run_plan(mf, layers, params, x, cut, grids, mf.BF16, plan_kwargs=dict(halo_reuse=True))
    refs = _oracle_groups(layers, params, x, cut, ("bf16_96", cut is None and 16 or cut))
    _check_groups(c, out, refs, cut, TOL_BF16)
    fixed = dict(force_nblk=32, force_mb=1)
    _, a = run_plan(mf, layers, params, x, cut, grids, mf.BF16, plan_kwargs=dict(halo_reuse=True, **fixed))
    _, b = run_plan(mf, layers, params, x, cut, grids, mf.BF16, plan_kwargs=fixed)
    assert np.array_equal(a, b)


def test_fp32_yolo16_96_halo_reuse(mf):
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 31, "fp32")
    x = synth.make_input(2, 96, 96, 3, 32, "fp32")
    c, out = run_plan(mf, layers, params, x, 8, [(3, 3), (2, 2)], mf.FP32, plan_kwargs=dict(halo_reuse=True))
    _check_groups(c, out, _oracle_groups(layers, params, x, 8, ("fp32_96", 8)), 8, TOL_FP32)


@pytest.mark.parametrize("name", ["yolo16_608_5x5_c8_2x2", "yolo25_608_5x5_c8_2x2"])
def test_bf16_608_halo_reuse(mf, name):
    wl = synth.workload(name)
    c, out = run_plan(mf, wl["layers"], wl["params"], wl["input"], wl["cut"], wl["grids"], mf.BF16,
                      plan_kwargs=dict(halo_reuse=True))
    _check_groups(c, out, _oracle_groups(wl["layers"], wl["params"], wl["input"], wl["cut"], name), wl["cut"],
                  TOL_BF16)


@pytest.mark.parametrize("cuts,grids", [([4, 8], [(3, 3), (2, 2), (2, 1)]), ([2, 6, 12], [(2, 2), (3, 2), (2, 2), (1, 2)])])
def test_bf16_yolo16_96_more_groups(mf, cuts, grids):
    # three and four layer groups (the outputs of groups 2.. are layer maps on the device):
    # the cut tensor and the output against the oracle, and bit-identical to a two-group
    # plan with fixed MMA shapes
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 41, "bf16")
    x = synth.make_input(2, 96, 96, 3, 42, "bf16")
    c, out = run_plan(mf, layers, params, x, cuts, grids, mf.BF16)
    refs = [oracle.group_outputs(layers, params, x[b], cuts) for b in range(2)]
    for b in range(2):
        assert rel_err(c[b], refs[b][0]) <= TOL_BF16 and rel_err(out[b], refs[b][-1]) <= TOL_BF16
    fixed = dict(force_nblk=32, force_mb=1)
    _, a = run_plan(mf, layers, params, x, cuts, grids, mf.BF16, plan_kwargs=fixed)
    _, e = run_plan(mf, layers, params, x, 8, [(2, 2), (1, 1)], mf.BF16, plan_kwargs=fixed)
    assert np.array_equal(a, e)


def test_fp32_yolo16_96_four_groups(mf):
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 31, "fp32")
    x = synth.make_input(2, 96, 96, 3, 32, "fp32")
    cuts = [2, 6, 12]
    c, out = run_plan(mf, layers, params, x, cuts, [(2, 2), (3, 2), (2, 2), (1, 2)], mf.FP32)
    for b in range(2):
        refs = oracle.group_outputs(layers, params, x[b], cuts)
        assert rel_err(c[b], refs[0]) <= TOL_FP32 and rel_err(out[b], refs[-1]) <= TOL_FP32


def test_bf16_608_three_groups(mf):
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, x = wl["layers"], wl["params"], wl["input"]
    cuts = [4, 8]
    c, out = run_plan(mf, layers, params, x, cuts, [(5, 5), (3, 3), (2, 2)], mf.BF16)
    outs = oracle.forward(layers, params, x[0])
    assert rel_err(c[0], outs[3]) <= TOL_BF16 and rel_err(out[0], outs[-1]) <= TOL_BF16


def test_measured_search_picks_the_fastest_timed_plan(mf):
    # Algorithm 2 re-targeted at the GPU: candidates whose intermediates fit the L2 are timed,
    # the others refused; the fastest is reported, and it computes the network correctly
    import torch
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    layers, params, x = wl["layers"], wl["params"], wl["input"]
    net = mf.Net(layers, 608, 608, 3)
    net.set_params(params)
    cands, best = net.search_measured(cuts=(8, 12), max_grid=3, runs=5)
    assert len(cands) == 3 + 2 * 9
    l2 = torch.cuda.get_device_properties(0).L2_cache_size
    for c in cands:
        if c["intermediate_bytes"] > l2:
            assert c["status"] == mf.ENOFIT and c["us_per_run"] is None
        else:
            assert c["status"] == mf.OK and c["us_per_run"] > 0
    timed = [i for i, c in enumerate(cands) if c["us_per_run"] is not None]
    assert best in timed
    assert cands[best]["us_per_run"] == min(cands[i]["us_per_run"] for i in timed)
    b = cands[best]
    _, out = run_plan(mf, layers, params, x, b["cut"], b["grids"], mf.BF16)
    assert rel_err(out[0], oracle.forward(layers, params, x[0])[-1]) <= TOL_BF16


@pytest.mark.parametrize("n_layers,cut,c,h,w,launches", [
    (8, 4, 3, 40, 56, 1),   # RGB rows of 336 bytes: widened in the kernel
    (4, 2, 3, 36, 44, 2),   # RGB rows of 264 bytes (not a multiple of 16): the layout kernel first
    (8, 4, 1, 32, 48, 1),   # one channel
    (8, 4, 5, 40, 40, 1),   # five channels
])
def test_bf16_nhwc_image_batch2(mf, n_layers, cut, c, h, w, launches):
    # the first layer reads the NHWC image of every frame in place (raw rows widened in the
    # kernel) or, for rows of another size, through the layout kernel; both at batch 2
    layers = synth.YOLO16[:n_layers]
    params = synth.make_params(layers, c, 71 + c, "bf16")
    x = synth.make_input(2, h, w, c, 72 + w, "bf16")
    net = mf.Net(layers, h, w, c)
    net.set_params(params)
    assert mf.Plan(net, cut, [(2, 3), (2, 2)], batch=2, dry_run=True).launches_per_run() == launches
    got_cut, out = run_plan(mf, layers, params, x, cut, [(2, 3), (2, 2)], mf.BF16)
    _check_groups(got_cut, out, _oracle_groups(layers, params, x, cut), cut, TOL_BF16)


# ---------------------------------------------------------------------------
# On-chip chaining of a 3x3 and the 1x1 after it (option chain=True: the 3x3's output stays in TMEM)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("cut,grids", [(8, [(3, 3), (2, 2)]), (6, [(2, 2), (2, 1)]), (None, [(3, 2)])])
def test_bf16_chained_pair_matches_unchained_and_oracle(mf, cut, grids):
    # YOLOv2 layers 4 -> 5 chained; with the cut after layer 5 the chained 1x1 writes the cut tensor
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 61, "bf16")
    x = synth.make_input(2, 96, 96, 3, 62, "bf16")
    c1, o1 = run_plan(mf, layers, params, x, cut, grids, mf.BF16, plan_kwargs=dict(chain=True))
    c0, o0 = run_plan(mf, layers, params, x, cut, grids, mf.BF16)
    assert np.array_equal(o1, o0)
    if cut is not None:
        assert np.array_equal(c1, c0)
    _check_groups(c1, o1, _oracle_groups(layers, params, x, cut), cut, TOL_BF16)


@pytest.mark.parametrize("layers", [
    [("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 32)],                        # chained 1x1 writes the output
    [("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 32), ("max", 2, 2, 0, 0)],   # ... through a fused max-pool
    [("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 48), ("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 16)],
])
def test_bf16_chained_pair_small_networks(mf, layers):
    params = synth.make_params(layers, 16, 63, "bf16")
    x = synth.make_input(2, 40, 48, 16, 64, "bf16")
    _, o1 = run_plan(mf, layers, params, x, None, [(2, 3)], mf.BF16, plan_kwargs=dict(chain=True))
    _, o0 = run_plan(mf, layers, params, x, None, [(2, 3)], mf.BF16)
    assert np.array_equal(o1, o0)
    _check_groups(None, o1, _oracle_groups(layers, params, x, None), None, TOL_BF16)


def test_bf16_608_chained_matches_unchained(mf):
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    c1, o1 = run_plan(mf, wl["layers"], wl["params"], wl["input"], 8, wl["grids"], mf.BF16,
                      plan_kwargs=dict(chain=True))
    c0, o0 = run_plan(mf, wl["layers"], wl["params"], wl["input"], 8, wl["grids"], mf.BF16)
    assert np.array_equal(o1, o0) and np.array_equal(c1, c0)


# ---------------------------------------------------------------------------
# Run paths: host buffers, CUDA graphs, repeated runs
# ---------------------------------------------------------------------------

def test_run_host_matches_device_run(mf):
    import torch
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    net = mf.Net(wl["layers"], 608, 608, 3)
    net.set_params(wl["params"])
    plan = mf.Plan(net, 8, wl["grids"], batch=1, dtype=mf.BF16)
    xin = torch.from_numpy(wl["input"]).to(torch.bfloat16)
    out_dev = torch.empty((1, 38, 38, 256), dtype=torch.bfloat16, device="cuda")
    plan.run(xin.cuda(), out_dev)
    plan.sync_status(like=out_dev)
    # the host call takes the same NHWC image from (pinned) host memory
    xh = torch.from_numpy(wl["input"]).to(torch.bfloat16).pin_memory()
    oh = torch.empty((1, 38, 38, 256), dtype=torch.bfloat16).pin_memory()
    plan.run_host(xh, oh)
    assert torch.equal(oh, out_dev.cpu())
    plan.run_host(xh, oh)  # staging buffers reused
    assert torch.equal(oh, out_dev.cpu())


def test_run_host_async_frames_in_flight_match_device_runs(mf):
    import torch
    wl = synth.workload("yolo16_416_1x3x3")
    net = mf.Net(wl["layers"], 416, 416, 3)
    net.set_params(wl["params"])
    plan = mf.Plan(net, None, wl["grids"], batch=1, dtype=mf.BF16)
    frames = [synth.make_input(1, 416, 416, 3, 100 + i) for i in range(3)]
    ref = []
    for x in frames:
        out = torch.empty((1, 26, 26, 256), dtype=torch.bfloat16, device="cuda")
        plan.run(torch.from_numpy(x).to(torch.bfloat16).cuda(), out)
        plan.sync_status(like=out)
        ref.append(out.cpu())
    xh = [torch.from_numpy(x).to(torch.bfloat16).pin_memory() for x in frames]
    oh = [torch.empty((1, 26, 26, 256), dtype=torch.bfloat16).pin_memory() for _ in frames]
    for i in range(3):  # three frames enqueued back to back over the two staging slots
        plan.run_host_async(xh[i], oh[i])
    plan.run_host_wait()
    for i in range(3):
        assert torch.equal(oh[i], ref[i]), i
    plan.run_host_wait()  # nothing in flight: returns at once


def test_run_host_fp32_matches_device_run(mf):
    import torch
    wl = synth.workload("tiny3_64_fp32")
    net = mf.Net(wl["layers"], wl["h"], wl["w"], 3)
    net.set_params(wl["params"])
    plan = mf.Plan(net, wl["cut"], wl["grids"], batch=wl["batch"], dtype=mf.FP32)
    sh = net.shape(len(wl["layers"]) - 1)
    xin = torch.from_numpy(wl["input"]).float()
    out_dev = torch.empty((wl["batch"], sh[3], sh[4], sh[5]), dtype=torch.float32, device="cuda")
    plan.run(xin.cuda(), out_dev)
    plan.sync_status(like=out_dev)
    xh = torch.from_numpy(wl["input"]).float().contiguous()
    oh = torch.empty(out_dev.shape, dtype=torch.float32)
    plan.run_host(xh, oh)
    assert torch.equal(oh, out_dev.cpu())


def test_cuda_graph_replay_matches(mf):
    import torch
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    net = mf.Net(wl["layers"], 608, 608, 3)
    net.set_params(wl["params"])
    plan = mf.Plan(net, 8, wl["grids"], batch=1, dtype=mf.BF16)
    xin = torch.from_numpy(wl["input"]).to(torch.bfloat16).cuda()
    out = torch.empty((1, 38, 38, 256), dtype=torch.bfloat16, device="cuda")
    plan.run(xin, out)
    plan.sync_status(like=xin)
    ref = out.clone()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        plan.run(xin, out, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    out.zero_()
    with torch.cuda.graph(g):
        plan.run(xin, out, stream=torch.cuda.current_stream())
    for _ in range(3):
        out.zero_()
        g.replay()
    torch.cuda.synchronize()
    plan.sync_status(like=xin)
    assert torch.equal(out, ref)


@pytest.mark.parametrize("dtype_name", ["BF16", "FP32"])
def test_unfinished_dependency_times_out_and_context_survives(mf, dtype_name):
    # Fault injection on the host side: one task's completion is never published,
    # so every tile waiting on it must give up after the short limit and the run
    # must report ETIMEOUT; the next run on the same context must succeed.
    import torch
    dt = getattr(mf, dtype_name)
    layers = synth.YOLO16
    params = synth.make_params(layers, 3, 51, "bf16")
    x = synth.make_input(1, 64, 64, 3, 52, "bf16")
    with pytest.raises(mf.MafatError) as e:
        run_plan(mf, layers, params, x, 8, [(2, 2), (2, 2)], dt,
                 plan_kwargs=dict(test_unpublished_task=0, wait_timeout_ns=50_000_000))
    assert e.value.status == 5
    c, out = run_plan(mf, layers, params, x, 8, [(2, 2), (2, 2)], dt)
    refs = _oracle_groups(layers, params, x, 8)
    _check_groups(c, out, refs, 8, TOL_BF16 if dt == mf.BF16 else TOL_FP32)
    torch.cuda.synchronize()
