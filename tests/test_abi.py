"""The C-ABI library loads and exports every entry point include/mafat.h declares (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "mafat.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"\b(mafat_[a-z_0-9]+)\s*\(", src)
    return sorted(set(names))


@pytest.fixture(scope="module")
def mf():
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    return mf


def test_header_declares_the_boundary_calls():
    """The three calls of the problem statement and the rest of the boundary: weights,
    status, debug run, region / predictor / search / statistics queries, cleanup."""
    names = _declared()
    for n in ("mafat_describe_net", "mafat_plan", "mafat_run", "mafat_set_weights", "mafat_sync_status",
              "mafat_run_debug", "mafat_tile_region", "mafat_predict_mem", "mafat_search", "mafat_plan_stats",
              "mafat_plan_destroy", "mafat_net_destroy", "mafat_last_error"):
        assert n in names, n


def test_library_exports_every_declared_symbol(mf):
    lib = ctypes.CDLL(mf.LIB_PATH)
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_covers_every_declared_symbol(mf):
    assert sorted(mf.EXPORTED) == _declared()


def test_version_and_error_strings(mf):
    assert "sm_103a" in mf.version()
    with pytest.raises(mf.MafatError) as e:
        mf.Net([("conv", 5, 1, 2, 16)], 8, 8, 3)
    assert e.value.status == 2  # EUNSUPPORTED
    assert "3x3" in str(e.value)


def test_run_refuses_dry_run_plans_without_touching_a_gpu(mf):
    import synth
    net = mf.Net(synth.TINY3, 16, 16, 3)
    net.set_params(synth.make_params(synth.TINY3, 3, 1, "fp32"))
    plan = mf.Plan(net, None, [(2, 2)], dry_run=True, dtype=mf.FP32)
    with pytest.raises(mf.MafatError) as e:
        plan.run(16, 4096)
    assert e.value.status == 1
