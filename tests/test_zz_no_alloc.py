"""mafat_run_fp32_noalloc: the allocation-free entry point, for callers that may not
allocate device memory while they run (global-mode stream capture, real-time loops
that forbid allocator calls, processes whose device memory another allocator owns).

It must give the same result as mafat_run on the same plan, on calls in a row and with
a differently shaped plan run through the shared static area in between (that area
keeps the previous call's contents), report a device-side wait timeout through
mafat_noalloc_sync_status, and refuse plans whose scratch does not fit its 32 MiB
area, bf16 plans and overlapping buffers, before launching anything.

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


def _setup(mf, layers, h, c, cut, grids, seed, batch=1, **plan_kwargs):
    import torch
    params = synth.make_params(layers, c, seed, "fp32")
    x = synth.make_input(batch, h, h, c, seed, "fp32")
    net = mf.Net(layers, h, h, c)
    net.set_params(params)
    plan = mf.Plan(net, cut, grids, batch=batch, dtype=mf.FP32, **plan_kwargs)
    xin = torch.from_numpy(x).cuda()  # NHWC
    sh = net.shape(len(layers) - 1)
    return net, plan, xin, (batch, sh[3], sh[4], sh[5])


def _case(mf, name):
    if name == "tiny3_64_2x2":
        return _setup(mf, synth.TINY3, 64, 3, None, [(2, 2)], synth.SEED_BASE)
    return _setup(mf, synth.YOLO16, 64, 3, 8, [(2, 2), (2, 2)], 77, batch=2)


def _reference(plan, xin, oshape):
    import torch
    ref = torch.empty(oshape, dtype=torch.float32, device="cuda")
    plan.run(xin, ref)
    plan.sync_status(like=xin)
    return ref.cpu().numpy()


def _noalloc(mf, plan, xin, oshape):
    import torch
    out = torch.full(oshape, float("nan"), dtype=torch.float32, device="cuda")
    plan.run_noalloc(xin, out)
    mf.Plan.noalloc_sync_status(like=xin)
    return out.cpu().numpy()


def _check(got, ref, what):
    assert np.isfinite(got).all(), "%s left outputs unwritten" % what
    err = float(np.abs(got - ref).max()) / float(np.abs(ref).max())
    assert err <= TOL_FP32, "%s: rel err %.3g" % (what, err)


@pytest.mark.parametrize("case", ["tiny3_64_2x2", "yolo16_64_cut8"])
def test_noalloc_matches_mafat_run_twice(mf, case):
    net, plan, xin, oshape = _case(mf, case)
    ref = _reference(plan, xin, oshape)
    for call in range(2):
        _check(_noalloc(mf, plan, xin, oshape), ref, "call %d" % call)


def test_noalloc_interleaved_plans_match_mafat_run(mf):
    # Two plans of different shapes take turns in the shared area, so each call finds
    # the other plan's tile buffers, cut tensor and counters left there.
    cases = [_case(mf, "tiny3_64_2x2"), _case(mf, "yolo16_64_cut8")]
    refs = [_reference(plan, xin, oshape) for _, plan, xin, oshape in cases]
    for step, k in enumerate([0, 1, 0, 1, 1, 0]):
        _, plan, xin, oshape = cases[k]
        _check(_noalloc(mf, plan, xin, oshape), refs[k], "step %d (plan %d)" % (step, k))


def test_noalloc_reports_a_wait_timeout_then_runs_clean(mf):
    # Fault injection on the host side: task 0's completion is never published, so the
    # tasks waiting on it give up after 50 ms and the status query reports ETIMEOUT.
    # The next call, with a normal plan, must run clean and match mafat_run.
    import torch
    _, bad, xin, oshape = _setup(mf, synth.YOLO16, 64, 3, 8, [(2, 2), (2, 2)], 78,
                                 test_unpublished_task=0, wait_timeout_ns=50_000_000)
    out = torch.zeros(oshape, dtype=torch.float32, device="cuda")
    bad.run_noalloc(xin, out)
    with pytest.raises(mf.MafatError) as e:
        mf.Plan.noalloc_sync_status(like=xin)
    assert e.value.status == mf.ETIMEOUT
    mf.Plan.noalloc_sync_status(like=xin)  # read once, then clear
    net, plan, xin2, oshape2 = _case(mf, "yolo16_64_cut8")
    ref = _reference(plan, xin2, oshape2)
    _check(_noalloc(mf, plan, xin2, oshape2), ref, "call after the timeout")


def test_noalloc_refuses_oversized_bf16_and_overlapping(mf):
    # Every refusal gets real device buffers of the plan's sizes, so that a regression
    # in the host-side checks could never launch a kernel on a bogus address.
    import torch
    layers = synth.YOLO16
    big = mf.Net(layers, 416, 416, 3)
    big.set_params(synth.make_params(layers, 3, 5, "fp32"))
    sh = big.shape(len(layers) - 1)
    xin = torch.zeros((1, 416, 416, 3), dtype=torch.float32, device="cuda")
    out = torch.zeros((1, sh[3], sh[4], sh[5]), dtype=torch.float32, device="cuda")
    plan = mf.Plan(big, None, [(3, 3)], dtype=mf.FP32)
    with pytest.raises(mf.MafatError) as e:
        plan.run_noalloc(xin, out)
    assert e.value.status == mf.EINVAL and "32 MiB" in str(e.value)
    bplan = mf.Plan(big, None, [(3, 3)], dtype=mf.BF16)
    with pytest.raises(mf.MafatError) as e:
        bplan.run_noalloc(xin.to(torch.bfloat16), out.to(torch.bfloat16))
    assert e.value.status == mf.EUNSUPPORTED
    _, small, xs, oshape = _case(mf, "tiny3_64_2x2")
    buf = torch.zeros(max(xs.numel(), int(np.prod(oshape))), dtype=torch.float32, device="cuda")
    with pytest.raises(mf.MafatError) as e:
        small.run_noalloc(buf, buf)
    assert e.value.status == mf.EINVAL and "overlap" in str(e.value)
    torch.cuda.synchronize()
