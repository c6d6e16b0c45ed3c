"""mafat_run_fp32_noalloc: the allocation-free entry point for callers that may not
allocate device memory while they run.  It must give the same result as mafat_run
on the same plan, on two calls in a row (the static scratch area keeps the previous
call's contents), and refuse plans whose scratch does not fit its 32 MiB area.

Collected last so that a stop at the first failure has run every other test first;
it also passes alone in a fresh process.
"""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

TOL_FP32 = 1e-4


@pytest.fixture(scope="module")
def mf():
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    return mf


def _setup(mf, layers, h, c, cut, grids, seed, batch=1):
    import torch
    params = synth.make_params(layers, c, seed, "fp32")
    x = synth.make_input(batch, h, h, c, seed, "fp32")
    net = mf.Net(layers, h, h, c)
    net.set_params(params)
    plan = mf.Plan(net, cut, grids, batch=batch, dtype=mf.FP32)
    xin = torch.from_numpy(mf.to_planar(x)).cuda()
    sh = net.shape(len(layers) - 1)
    return net, plan, xin, (batch, sh[3], sh[4], sh[5])


@pytest.mark.parametrize("case", ["tiny3_64_2x2", "yolo16_64_cut8"])
def test_noalloc_matches_mafat_run_twice(mf, case):
    import torch
    if case == "tiny3_64_2x2":
        net, plan, xin, oshape = _setup(mf, synth.TINY3, 64, 3, None, [(2, 2)], synth.SEED_BASE)
    else:
        net, plan, xin, oshape = _setup(mf, synth.YOLO16, 64, 3, 8, [(2, 2), (2, 2)], 77, batch=2)
    ref = torch.empty(oshape, dtype=torch.float32, device="cuda")
    plan.run(xin, ref)
    plan.sync_status(like=xin)
    ref_np = ref.cpu().numpy()
    den = float(np.abs(ref_np).max())
    for call in range(2):
        out = torch.full(oshape, float("nan"), dtype=torch.float32, device="cuda")
        plan.run_noalloc(xin, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.isfinite(got).all(), "call %d left outputs unwritten" % call
        err = float(np.abs(got - ref_np).max()) / den
        assert err <= TOL_FP32, "call %d: rel err %.3g" % (call, err)


def test_noalloc_refuses_oversized_and_bf16_plans(mf):
    layers = synth.YOLO16
    big = mf.Net(layers, 416, 416, 3)
    big.set_params(synth.make_params(layers, 3, 5, "fp32"))
    plan = mf.Plan(big, None, [(3, 3)], dtype=mf.FP32)
    with pytest.raises(mf.MafatError) as e:
        plan.run_noalloc(16, 16)
    assert e.value.status == 1 and "32 MiB" in str(e.value)
    bplan = mf.Plan(big, None, [(3, 3)], dtype=mf.BF16)
    with pytest.raises(mf.MafatError) as e:
        bplan.run_noalloc(16, 16)
    assert e.value.status == 2
