"""Tensor-core operand / accumulator layouts the kernels rely on (runs first among the GPU tests).

One 128 x n x 16 bf16 MMA through mafat_diag_umma, against a float64 product.
Both assignments of the shared-memory descriptor's two offset fields are run
(the diagnostic's operand layout keeps both inside its buffers); exactly the one
the kernels are compiled with must reproduce A * B^T.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mf():
    import __graft_entry__ as g
    g.build()
    import paper_2107_06960_gb300 as mf
    return mf


def _product(mf, n, lbo_is_k, seed):
    import torch
    rng = np.random.default_rng(seed)
    a = rng.standard_normal((128, 16)).astype(np.float32)
    b = rng.standard_normal((n, 16)).astype(np.float32)
    at = torch.from_numpy(a).to(torch.bfloat16).cuda()
    bt = torch.from_numpy(b).to(torch.bfloat16).cuda()
    d = torch.zeros((128, n), dtype=torch.float32, device="cuda")
    mf.diag_umma(at, bt, d, n, lbo_is_k)
    torch.cuda.synchronize()
    ref = at.double().cpu().numpy() @ bt.double().cpu().numpy().T
    return d.cpu().numpy(), ref


@pytest.mark.parametrize("n", [16, 32, 64, 128, 256])
def test_umma_bf16_product_and_tmem_layout(mf, n):
    got, ref = _product(mf, n, 1, n)
    np.testing.assert_allclose(got, ref, rtol=1e-5, atol=1e-5)


def test_other_descriptor_field_assignment_is_wrong(mf):
    got, ref = _product(mf, 64, 0, 7)
    assert not np.allclose(got, ref, rtol=1e-3, atol=1e-3)
