import os
"""Host planner of the C ABI (shapes, Grid regions, Algorithms 1-2, work tables) against the oracle.

All on the CPU: network queries need no device, and plans are built with
dry_run so that no device memory is touched.
"""
import numpy as np
import pytest

import oracle
import synth


@pytest.fixture(scope="module")
def mf():
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    return mf


def _net(mf, layers, size, c=3, dtype="bf16", seed=1):
    net = mf.Net(layers, size, size, c)
    net.set_params(synth.make_params(layers, c, seed, dtype))
    return net


@pytest.mark.parametrize("size", [608, 416, 1216, 64, 96])
def test_shapes_match_oracle(mf, size):
    net = _net(mf, synth.YOLO16, size)
    ref = oracle.layer_shapes(synth.YOLO16, size, size, 3)
    for l, sh in enumerate(ref):
        assert net.shape(l) == (sh["h_in"], sh["w_in"], sh["c_in"], sh["h_out"], sh["w_out"], sh["c_out"])


@pytest.mark.parametrize("size,first,last,n,m", [
    (608, 0, 7, 5, 5), (608, 8, 15, 2, 2), (416, 0, 15, 3, 3), (1216, 0, 7, 8, 8), (1216, 8, 15, 4, 4),
    (608, 0, 1, 5, 5), (608, 2, 15, 3, 2), (64, 0, 11, 5, 5), (96, 12, 15, 4, 3), (608, 0, 15, 7, 1)])
def test_tile_regions_match_oracle(mf, size, first, last, n, m):
    layers = synth.YOLO16
    net = _net(mf, layers, size)
    shapes = oracle.layer_shapes(layers, size, size, 3)
    for i in range(n):
        for j in range(m):
            ref = oracle.tile_regions(layers, shapes, (first, last), n, m, i, j)
            for l in range(first, last + 1):
                out_r, in_r = net.tile_region(first, last, n, m, i, j, l)
                if ref[l][0][1] <= ref[l][0][0] or ref[l][0][3] <= ref[l][0][2]:
                    assert out_r[1] <= out_r[0] or out_r[3] <= out_r[2]
                    continue
                assert out_r == ref[l][0] and in_r == ref[l][1]


@pytest.mark.parametrize("size", [608, 416])
def test_predictor_matches_oracle_exactly(mf, size):
    layers = synth.YOLO16
    net = _net(mf, layers, size)
    shapes = oracle.layer_shapes(layers, size, size, 3)
    for cut in (None, 2, 4, 8, 12):
        for t1 in range(1, 6):
            for t2 in (1, 2, 3):
                grids = [(t1, t1)] if cut is None else [(t1, t1), (t2, t2)]
                ref = oracle.predict_mem(layers, shapes, cut, grids)
                got = net.predict_mem(cut if cut is not None else 16, t1, t1, t2, t2)
                assert got == ref
    for first, last in ((0, 15), (0, 7), (8, 15), (2, 2)):
        for f in (1, 2):
            ref = oracle.predict_layer_group(layers, shapes, (first, last), 3, 2, 31.0, input_factor=f)
            assert net.predict_layer_group(first, last, 3, 2, 31.0, f) == ref


def test_predictor_matches_hand_computed_tiled_case(mf):
    # the library's Algorithm 1 on the hand-worked 2x2 case of tests/golden/alg1_tiled_2x2.txt
    layers = [("conv", 3, 1, 1, 8), ("max", 2, 2, 0, 0), ("conv", 3, 1, 1, 16)]
    net = mf.Net(layers, 18, 14, 4)
    mx = {}
    with open(os.path.join(os.path.dirname(__file__), "golden", "alg1_tiled_2x2.txt")) as fh:
        for line in fh:
            if line.startswith("max_mem_elements"):
                mx[line.split()[0]] = int(line.split()[1])
    assert net.predict_layer_group(0, 2, 2, 2, 0.0, 2) == mx["max_mem_elements"] * 4 / 2 ** 20
    assert net.predict_layer_group(0, 2, 2, 1, 0.0, 2) == mx["max_mem_elements_2x1"] * 4 / 2 ** 20
    assert net.predict_layer_group(0, 2, 1, 2, 0.0, 2) == mx["max_mem_elements_1x2"] * 4 / 2 ** 20
    for (i, j) in ((0, 0), (1, 1)):
        out_r, in_r = net.tile_region(0, 2, 2, 2, i, j, 0)
        ref = oracle.tile_regions(layers, oracle.layer_shapes(layers, 18, 14, 4), (0, 2), 2, 2, i, j)[0]
        assert out_r == ref[0] and in_r == ref[1]


def test_search_matches_oracle_for_table1_limits(mf):
    layers = synth.YOLO16
    net = _net(mf, layers, 608)
    shapes = oracle.layer_shapes(layers, 608, 608, 3)
    for limit in (256, 192, 128, 96, 80, 64, 48, 32, 16, 1000, 1):
        assert net.search(float(limit)) == oracle.get_config(layers, shapes, float(limit))


def _region_flops(layers, size, cut, grids, batch):
    shapes = oracle.layer_shapes(layers, size, size, 3)
    tot = 0
    for g, (n, m) in zip(oracle.groups_of(len(layers), cut), grids):
        for i in range(n):
            for j in range(m):
                regs = oracle.tile_regions(layers, shapes, g, n, m, i, j)
                for l in range(g[0], g[1] + 1):
                    t, k, s, p, f = layers[l]
                    if t != "conv":
                        continue
                    (y0, y1, x0, x1), _ = regs[l]
                    tot += 2 * max(y1 - y0, 0) * max(x1 - x0, 0) * f * shapes[l]["c_in"] * k * k
    return tot * batch


@pytest.mark.parametrize("name", ["yolo16_416_1x3x3", "yolo16_608_5x5_c8_2x2", "yolo16_1216_b8_8x8_c8_4x4",
                                  "yolo25_608_5x5_c8_2x2"])
def test_plan_statistics(mf, name):
    wl = synth.WORKLOADS[name]
    layers, size, batch = wl["layers"], wl["h"], wl["batch"]
    net = _net(mf, layers, size)
    plan = mf.Plan(net, wl["cut"], wl["grids"], batch=batch, dtype=mf.BF16, dry_run=True)
    st = plan.stats()
    shapes = oracle.layer_shapes(layers, size, size, 3)
    assert st["useful_flops"] == oracle.conv_flops(layers, shapes) * batch
    assert st["executed_flops"] == _region_flops(layers, size, wl["cut"], wl["grids"], batch)
    assert st["issued_flops"] >= st["executed_flops"] >= st["useful_flops"]
    ref_pred = oracle.predict_mem(layers, shapes, wl["cut"], wl["grids"])
    assert st["predicted_mib"] == ref_pred
    ntiles = sum(n * m for n, m in wl["grids"][:1 if wl["cut"] is None else 2])
    assert st["n_tiles"] == ntiles * batch


def test_headline_plan_numbers(mf):
    # 608x608, cut after layer 7, 5x5 / 2x2: 26.0 GFLOP useful, 13.7 % halo recompute
    wl = synth.WORKLOADS["yolo16_608_5x5_c8_2x2"]
    net = _net(mf, wl["layers"], 608)
    st = mf.Plan(net, 8, wl["grids"], dry_run=True).stats()
    assert abs(st["useful_flops"] / 1e9 - 26.0007) < 1e-3
    assert abs(st["executed_flops"] / st["useful_flops"] - 1.137) < 0.01


def test_flat_blocks_cut_block_padding(mf):
    # 38x38 on a 2x2 grid gives 19x19 conv regions: 2 x 3 rectangles of 16x8 pixels, or the
    # region's rows laid end to end at a pitch of 24 pixels (19 + 2 halo, rounded up to 8):
    # 19 * 24 = 456 pixels, 4 runs of 128
    conv = [("conv", 3, 1, 1, 512)]
    net = mf.Net(conv, 38, 38, 256)
    net.set_params(synth.make_params(conv, 256, 1, "bf16"))
    flat = mf.Plan(net, None, [(2, 2)], dry_run=True).stats()
    rect = mf.Plan(net, None, [(2, 2)], dry_run=True, rect_blocks=True).stats()
    mac = 2 * 128 * 512 * 256 * 9
    assert flat["issued_flops"] == 4 * 4 * mac and rect["issued_flops"] == 4 * 6 * mac
    assert flat["executed_flops"] == rect["executed_flops"] == 38 * 38 * 512 * 256 * 9 * 2
    # a convolution with a fused pool keeps its rectangles (a window's pixels must share a warp)
    pooled = [("conv", 3, 1, 1, 64), ("max", 2, 2, 0, 0)]
    net = mf.Net(pooled, 76, 76, 128)
    net.set_params(synth.make_params(pooled, 128, 1, "bf16"))
    assert (mf.Plan(net, None, [(2, 2)], dry_run=True).stats()["issued_flops"] ==
            mf.Plan(net, None, [(2, 2)], dry_run=True, rect_blocks=True).stats()["issued_flops"])
    # the benchmark plan: layers 12-15 (19-20 pixel regions) go from 24 blocks to 16 each
    wl = synth.WORKLOADS["yolo16_608_5x5_c8_2x2"]
    net = _net(mf, wl["layers"], 608)
    a = mf.Plan(net, 8, wl["grids"], dry_run=True).stats()["issued_flops"]
    b = mf.Plan(net, 8, wl["grids"], dry_run=True, rect_blocks=True).stats()["issued_flops"]
    saved = 8 * 128 * 2 * (2 * 512 * 256 * 9 + 2 * 256 * 512)
    assert b - a == saved


@pytest.mark.parametrize("c, k_issued", [(1, 48), (3, 48), (4, 48), (5, 80), (8, 80)])
def test_first_layer_k_steps(mf, c, k_issued):
    # A 3x3 first layer of c < 8 channels read from the NHWC image: up to 4 channels go in
    # pixel pairs (a 16-byte halo slot holds two pixels, one K = 16 step covers a kernel row:
    # 3 steps, K 48); 5-7 channels pair taps over 8-channel pixels (5 steps, K 80), and so do
    # 8-channel inputs read as one octet plane.  64x64 on one tile: 4 x 8 blocks of 16x8.
    conv = [("conv", 3, 1, 1, 32)]
    net = mf.Net(conv, 64, 64, c)
    net.set_params(synth.make_params(conv, c, 1, "bf16"))
    st = mf.Plan(net, None, [(1, 1)], dry_run=True).stats()
    assert st["issued_flops"] == 2 * (4 * 8 * 128) * 32 * k_issued
    assert st["executed_flops"] == 2 * 64 * 64 * 32 * c * 9
    # the fp32 check mode has no tensor-core packing: issued = executed
    st32 = mf.Plan(net, None, [(1, 1)], dtype=mf.FP32, dry_run=True).stats()
    assert st32["executed_flops"] == st["executed_flops"]


def test_gathered_first_layer_packs_blocks_across_columns(mf):
    # The first layer read from the RGB image keeps one halo per block, so an item's blocks
    # are any run of its task's blocks in column-major order: a 144x1216 map on one tile is
    # 9 block rows x 152 block columns = 1368 blocks, enough for 8 blocks per item on 152
    # CTAs: 171 items of 8 (stacked per block column it takes 2 items per column, 304).  A
    # first layer of 8 channels is read as an octet plane and keeps stacked blocks.
    conv = [("conv", 3, 1, 1, 32)]
    for c, items in ((3, 171), (8, 304)):
        net = mf.Net(conv, 144, 1216, c)
        net.set_params(synth.make_params(conv, c, 1, "bf16"))
        st = mf.Plan(net, None, [(1, 1)], dry_run=True).stats()
        assert st["n_items"] == items, (c, st["n_items"])
        assert st["issued_flops"] == 2 * 1368 * 128 * 32 * (48 if c == 3 else 80)
    # with the pool fused the blocks and items are the same
    pooled = [("conv", 3, 1, 1, 32), ("max", 2, 2, 0, 0)]
    net = mf.Net(pooled, 144, 1216, 3)
    net.set_params(synth.make_params(pooled, 3, 1, "bf16"))
    assert mf.Plan(net, None, [(1, 1)], dry_run=True).stats()["n_items"] == 171


def test_plan_validation_errors(mf):
    layers = synth.YOLO16
    net = _net(mf, layers, 64)
    with pytest.raises(mf.MafatError) as e:     # cut between a conv and its max-pool
        mf.Plan(net, 1, [(2, 2), (2, 2)], dry_run=True)
    assert e.value.status == 2
    with pytest.raises(mf.MafatError) as e:
        mf.Plan(net, 16, [(2, 2), (2, 2)], dry_run=True)
    assert e.value.status == 1
    with pytest.raises(mf.MafatError) as e:
        mf.Plan(net, None, [(0, 2)], dry_run=True)
    assert e.value.status == 1
    bare = mf.Net(layers, 64, 64, 3)             # weights never set
    with pytest.raises(mf.MafatError) as e:
        mf.Plan(bare, None, [(1, 1)], dry_run=True)
    assert e.value.status == 1
    with pytest.raises(mf.MafatError) as e:      # odd map under a max-pool
        mf.Net(layers, 66, 66, 3)
    assert e.value.status == 2


def test_grid_finer_than_output_skips_empty_tiles(mf):
    layers = synth.YOLO16
    net = _net(mf, layers, 64)
    # group 1 output at cut 12 is 4x4; a 5x5 grid has empty rows/columns of tiles
    st = mf.Plan(net, 12, [(5, 5), (3, 3)], dry_run=True).stats()
    assert st["n_tiles"] == 4 * 4 + 3 * 3


def test_measured_search_dry_run_candidates(mf):
    # the candidate list of the measured search (Algorithm 2 re-targeted at the GPU): order,
    # sizes, the L2 budget rule and the non-square grids, all on the host
    net = _net(mf, synth.YOLO16, 608)
    cands, best = net.search_measured(dry_run=True, budget_bytes=-1)
    assert best == -1
    assert len(cands) == 5 + 4 * 25
    assert [c["grids"] for c in cands[:5]] == [[(t, t)] for t in range(1, 6)]
    assert all(c["n_groups"] == 1 and c["cut"] is None for c in cands[:5])
    assert [c["cut"] for c in cands[5:]] == [cut for cut in (2, 4, 8, 12) for _ in range(25)]
    assert [c["grids"] for c in cands[5:30]] == [[(a, a), (b, b)] for a in range(1, 6) for b in range(1, 6)]
    for c in cands[::7]:
        st = mf.Plan(net, c["cut"], c["grids"], dry_run=True).stats()
        cut_bytes = 0
        if c["cut"] is not None:
            sh = net.shape(c["cut"] - 1)
            cut_bytes = (sh[5] + 7) // 8 * 8 * sh[3] * sh[4] * 2
        assert c["intermediate_bytes"] == st["scratch_bytes"] + cut_bytes
        assert c["predicted_mib"] == st["predicted_mib"]
        assert c["executed_flops"] == st["executed_flops"]
        assert c["status"] == 0 and c["us_per_run"] is None
    # with a budget, exactly the candidates above it are refused (MAFAT_ENOFIT)
    budget = sorted(c["intermediate_bytes"] for c in cands)[len(cands) // 2]
    capped, _ = net.search_measured(dry_run=True, budget_bytes=budget)
    assert [c["status"] for c in capped] == [
        mf.ENOFIT if c["intermediate_bytes"] > budget else 0 for c in cands]
    # non-square tilings: N x M with |N - M| <= 1, 13 per group
    ns, _ = net.search_measured(dry_run=True, square_only=False, cuts=(8,), budget_bytes=-1)
    assert len(ns) == 13 + 13 * 13
    assert all(abs(n - m) <= 1 for c in ns for n, m in c["grids"])
    assert (5, 4) in [c["grids"][0] for c in ns[:13]]


def test_tile_regions_with_explicit_bounds_match_oracle(mf):
    # a non-uniform tiling passed as tile bounds: every tile's regions equal the oracle's
    layers = synth.YOLO16
    net = _net(mf, layers, 608)
    shapes = oracle.layer_shapes(layers, 608, 608, 3)
    bounds = [([0, 20, 30, 45, 60, 76], [0, 12, 30, 50, 64, 76]), ([0, 15, 38], [0, 24, 38])]
    plan = mf.Plan(net, 8, [(5, 5), (2, 2)], dry_run=True, tile_bounds=bounds)
    for gi, g in enumerate(oracle.groups_of(len(layers), 8)):
        rb, cb = bounds[gi]
        for i in range(len(rb) - 1):
            for j in range(len(cb) - 1):
                ref = oracle.tile_regions(layers, shapes, g, len(rb) - 1, len(cb) - 1, i, j, (rb, cb))
                for l in range(g[0], g[1] + 1):
                    assert plan.tile_region(gi, i, j, l) == ref[l], (gi, i, j, l)
    with pytest.raises(mf.MafatError):   # bounds must increase strictly and cover the map
        mf.Plan(net, 8, [(5, 5), (2, 2)], dry_run=True,
                tile_bounds=[([0, 20, 20, 45, 60, 76], bounds[0][1]), bounds[1]])
    with pytest.raises(mf.MafatError):
        mf.Plan(net, 8, [(5, 5), (2, 2)], dry_run=True, tile_bounds=[([0, 20, 30, 45, 76], bounds[0][1]), bounds[1]])


def _band_work(layers, shapes, group, axis, lo, hi):
    """Executed MACs of the band [lo, hi) of the group's output along `axis`, the other
    axis whole, through the oracle's Grid traversal."""
    first, last = group
    sh = shapes[last]
    size = sh["h_out"] if axis == 0 else sh["w_out"]
    band = sorted({0, lo, hi, size})          # a partition with [lo, hi) as one of its parts
    k = band.index(lo)
    whole = [0, sh["w_out"] if axis == 0 else sh["h_out"]]
    b = (band, whole) if axis == 0 else (whole, band)
    n, m = (len(band) - 1, 1) if axis == 0 else (1, len(band) - 1)
    regs = oracle.tile_regions(layers, shapes, group, n, m, *((k, 0) if axis == 0 else (0, k)), b)
    w = 0
    for l in range(first, last + 1):
        t, k, s, p, f = layers[l]
        if t == oracle.CONV:
            (y0, y1, x0, x1), _ = regs[l]
            w += (y1 - y0) * (x1 - x0) * shapes[l]["c_out"] * shapes[l]["c_in"] * k * k
    return w


@pytest.mark.parametrize("group,n", [((8, 15), 4), ((0, 15), 5), ((0, 7), 3), ((4, 11), 3)])
def test_balanced_bounds_minimise_the_largest_part(mf, group, n):
    # the work-balanced non-uniform tiling against exhaustive search over every partition
    import itertools
    layers = synth.YOLO16
    net = _net(mf, layers, 608)
    shapes = oracle.layer_shapes(layers, 608, 608, 3)
    length = shapes[group[1]]["h_out"]
    rows, cols = net.balanced_bounds(group[0], group[1], n, n)
    assert rows == cols  # square map, same rule per axis
    assert rows[0] == 0 and rows[-1] == length and all(a < b for a, b in zip(rows, rows[1:]))
    work = {(a, b): _band_work(layers, shapes, group, 0, a, b) for a in range(length) for b in range(a + 1, length + 1)}
    got = max(work[(a, b)] for a, b in zip(rows, rows[1:]))
    best = min(max(work[(a, b)] for a, b in zip((0,) + cuts, cuts + (length,)))
               for cuts in itertools.combinations(range(1, length), n - 1))
    assert got == best
    even = oracle.grid_bounds(length, n)
    assert got <= max(work[r] for r in even)


@pytest.mark.parametrize("cut,grids", [(None, [(5, 5)]), (2, [(4, 4), (3, 3)]), (8, [(5, 5), (2, 2)]),
                                       (12, [(3, 2), (2, 3)])])
def test_halo_reuse_plan_computes_each_pixel_once(mf, cut, grids):
    # inter-tile reuse: every tile owns a part of every layer (the group-output tile scaled
    # through the pools), the parts partition each map, and nothing is recomputed
    layers = synth.YOLO16
    net = _net(mf, layers, 608)
    shapes = oracle.layer_shapes(layers, 608, 608, 3)
    plan = mf.Plan(net, cut, grids, dry_run=True, halo_reuse=True)
    st = plan.stats()
    assert st["executed_flops"] == st["useful_flops"]
    for gi, g in enumerate(oracle.groups_of(len(layers), cut)):
        n, m = grids[gi]
        for l in range(g[0], g[1] + 1):
            cover = np.zeros((shapes[l]["h_out"], shapes[l]["w_out"]), dtype=np.int64)
            for i in range(n):
                for j in range(m):
                    (oy0, oy1, ox0, ox1), (iy0, iy1, ix0, ix1) = plan.tile_region(gi, i, j, l)
                    cover[oy0:oy1, ox0:ox1] += 1
                    t, k, s, p, f = layers[l]
                    # the input region is the owned part's receptive field, clipped to the map
                    if oy1 > oy0 and ox1 > ox0:
                        assert (iy0, iy1) == (max(oy0 * s - p, 0), min((oy1 - 1) * s - p + k, shapes[l]["h_in"]))
                        assert (ix0, ix1) == (max(ox0 * s - p, 0), min((ox1 - 1) * s - p + k, shapes[l]["w_in"]))
            assert np.all(cover == 1), (g, l)


@pytest.mark.parametrize("cuts,grids", [([4, 8], [(5, 5), (3, 3), (2, 2)]), ([2, 6, 12], [(4, 4), (3, 3), (2, 2), (1, 1)])])
def test_plan_with_more_groups(mf, cuts, grids):
    # three and four layer groups: regions, executed work and group I/O as the oracle's
    layers = synth.YOLO16
    net = _net(mf, layers, 608)
    plan = mf.Plan(net, cuts, grids, dry_run=True)
    st = plan.stats()
    assert st["n_groups"] == len(cuts) + 1
    assert st["executed_flops"] == _region_flops(layers, 608, cuts, grids, 1)
    shapes = oracle.layer_shapes(layers, 608, 608, 3)
    for gi, g in enumerate(oracle.groups_of(len(layers), cuts)):
        n, m = grids[gi]
        for i in range(n):
            for j in range(m):
                ref = oracle.tile_regions(layers, shapes, g, n, m, i, j)
                for l in (g[0], g[1]):
                    assert plan.tile_region(gi, i, j, l) == ref[l]
    planar = lambda l: (shapes[l]["c_out"] + 7) // 8 * 8 * shapes[l]["h_out"] * shapes[l]["w_out"]
    io = 3 * 608 * 608 + shapes[15]["h_out"] * shapes[15]["w_out"] * shapes[15]["c_out"]  # NHWC image, output
    io += sum(2 * planar(c - 1) for c in cuts)
    assert st["group_io_bytes"] == io * 2
    with pytest.raises(mf.MafatError):
        mf.Plan(net, [8, 4], [(2, 2)] * 3, dry_run=True)      # cuts must increase
    with pytest.raises(mf.MafatError):
        mf.Plan(net, [2, 4, 8, 12], [(2, 2)] * 5, dry_run=True)  # at most four groups


def test_frames_in_flight_plan(mf):
    # batch > 1 with two groups: the ring spans one frame's 25 + 4 tiles and the hand-out
    # order overlaps frame f's second group with frame f + 1's first (the planner's own
    # check then guarantees every dependency points to an earlier item); the tasks and
    # the work per frame are those of batch 1 (1x1 layers take wider output-channel
    # blocks, hence fewer items), and the overlap is only taken where it is safe
    wl = synth.WORKLOADS["yolo16_608_5x5_c8_2x2"]
    net = _net(mf, wl["layers"], 608)
    one = mf.Plan(net, 8, wl["grids"], dry_run=True).stats()
    assert one["frames_overlapped"] == 0
    for k in (2, 3, 5):
        st = mf.Plan(net, 8, wl["grids"], batch=k, dry_run=True).stats()
        assert st["frames_overlapped"] == 1 and st["ring_slots"] == 29
        assert st["n_tasks"] == k * one["n_tasks"] and st["n_items"] < k * one["n_items"]
        assert abs(st["executed_flops"] - k * one["executed_flops"]) < 1e-3 * st["executed_flops"]
        fm = mf.Plan(net, 8, wl["grids"], batch=k, dry_run=True, frame_major=True).stats()
        assert fm["frames_overlapped"] == 0 and fm["n_items"] == st["n_items"]
    # not taken: one group, halo reuse, or a ring too small for a whole frame
    assert mf.Plan(net, None, [(3, 3)], batch=2, dry_run=True).stats()["frames_overlapped"] == 0
    assert mf.Plan(net, 8, wl["grids"], batch=2, dry_run=True, halo_reuse=True).stats()["frames_overlapped"] == 0
    assert mf.Plan(net, 8, wl["grids"], batch=2, dry_run=True, ring_slots=25).stats()["frames_overlapped"] == 0
    big = synth.WORKLOADS["yolo16_1216_b8_8x8_c8_4x4"]
    net2 = _net(mf, big["layers"], 1216)
    st = mf.Plan(net2, 8, big["grids"], batch=2, dry_run=True).stats()
    assert st["frames_overlapped"] == 1 and st["ring_slots"] == 80  # 64 + 16 tiles per frame
    assert mf.Plan(net2, 8, big["grids"], dry_run=True).stats()["ring_slots"] == 64  # one frame: 64 tiles


@pytest.mark.parametrize("cut", [2, 4, 8, 12])
@pytest.mark.parametrize("grids", [[(1, 1), (1, 1)], [(5, 5), (2, 2)], [(2, 2), (5, 5)], [(3, 4), (4, 3)]])
def test_frames_in_flight_every_cut_and_grid(mf, cut, grids):
    # the overlapped hand-out order is built (and passes the planner's dependency check)
    # for every cut and tiling, with the tasks of batch 1 once per frame
    net = _net(mf, synth.YOLO16, 96)
    one = mf.Plan(net, cut, grids, dry_run=True).stats()
    st = mf.Plan(net, cut, grids, batch=3, dry_run=True).stats()
    assert st["frames_overlapped"] == 1
    assert st["n_tasks"] == 3 * one["n_tasks"]
    assert abs(st["executed_flops"] - 3 * one["executed_flops"]) < 1e-6 * st["executed_flops"]


@pytest.mark.parametrize("c,w,launches", [(3, 608, 1), (3, 40, 1), (3, 28, 2), (4, 34, 1), (1, 20, 2), (8, 22, 1),
                                          (16, 18, 2)])
def test_input_layout_needs_no_conversion_when_rows_allow(mf, c, w, launches):
    # mafat_run reads an NHWC image in place (raw rows widened inside the kernel) whenever
    # a raw image row is a multiple of 16 bytes, 8 channels as they are; otherwise (and for
    # inputs of more than 8 channels) a layout kernel runs first
    layers = [("conv", 3, 1, 1, 16)]
    net = mf.Net(layers, 16, w, c)
    net.set_params(synth.make_params(layers, c, 3, "bf16"))
    plan = mf.Plan(net, None, [(1, 1)], dtype=mf.BF16, dry_run=True)
    assert plan.launches_per_run() == launches
    assert plan.stats()["group_io_bytes"] == 2 * (16 * w * c + 16 * w * 16)
    fplan = mf.Plan(net, None, [(1, 1)], dtype=mf.FP32, dry_run=True)
    assert fplan.launches_per_run() == 1


def test_chained_pairs_in_the_benchmark_plan(mf):
    # with chain=True, bf16 plans run a 3x3 convolution and the 1x1 after it in one item where
    # both fit one TMEM accumulator buffer (YOLOv2 layers 4 -> 5: 128 + 64 + 64 columns): one
    # task per tile fewer, the same regions and the same work
    wl = synth.workload("yolo16_608_5x5_c8_2x2")
    net = _net(mf, wl["layers"], 608)
    chained = mf.Plan(net, 8, wl["grids"], dry_run=True, chain=True)
    plain = mf.Plan(net, 8, wl["grids"], dry_run=True)
    a, b = chained.stats(), plain.stats()
    assert b["n_tasks"] - a["n_tasks"] == 25  # layer 5 of each group-1 tile
    assert a["executed_flops"] == b["executed_flops"] and a["issued_flops"] == b["issued_flops"]
    for i, j in ((0, 0), (2, 3), (4, 4)):
        for l in (4, 5, 6):
            assert chained.tile_region(0, i, j, l) == plain.tile_region(0, i, j, l)
    # fp32 plans and halo-reuse plans keep every convolution a stage of its own
    f32 = mf.Plan(net, 8, wl["grids"], dry_run=True, dtype=mf.FP32, chain=True)
    assert f32.stats()["n_tasks"] == b["n_tasks"]
    hr_c = mf.Plan(net, 8, wl["grids"], dry_run=True, halo_reuse=True, chain=True)
    hr_p = mf.Plan(net, 8, wl["grids"], dry_run=True, halo_reuse=True)
    assert hr_c.stats()["n_tasks"] == hr_p.stats()["n_tasks"]


@pytest.mark.parametrize("layers,chained", [
    ([("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 32)], 1),                    # 64 + 32 + 32 columns
    ([("conv", 3, 1, 1, 64), ("conv", 1, 1, 0, 32), ("max", 2, 2, 0, 0)], 1),
    ([("conv", 3, 1, 1, 128), ("conv", 1, 1, 0, 128)], 0),                  # 128 + 64 + 128 > 256
    ([("conv", 3, 1, 1, 64), ("max", 2, 2, 0, 0), ("conv", 1, 1, 0, 32)], 0),  # pool in between
    ([("conv", 3, 1, 1, 32), ("conv", 1, 1, 0, 32)], 0),                    # 3x3 output not a multiple of 64
])
def test_chain_eligibility(mf, layers, chained):
    net = mf.Net(layers, 32, 32, 16)
    net.set_params(synth.make_params(layers, 16, 9, "bf16"))
    c = mf.Plan(net, None, [(2, 2)], dry_run=True, chain=True).stats()
    p = mf.Plan(net, None, [(2, 2)], dry_run=True).stats()
    assert p["n_tasks"] - c["n_tasks"] == 4 * chained
