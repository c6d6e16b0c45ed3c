"""Tensor-core operand / accumulator layouts the kernels rely on (runs first among the GPU tests).

One 128 x n x 16 bf16 MMA through mafat_diag_umma, with the fused kernel's
shared-memory descriptor encoding and TMEM accumulator layout, against a float64
product of the same bf16 operands; A is read from shared memory, or from tensor memory
(two bf16 per 32-bit column, lane = row) as chained 3x3 -> 1x1 layers pass it.
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


@pytest.mark.parametrize("a_in_tmem", [False, True])
@pytest.mark.parametrize("n", [16, 32, 64, 128, 256])
def test_umma_bf16_product_and_tmem_layout(mf, n, a_in_tmem):
    import torch
    rng = np.random.default_rng(n)
    a = rng.standard_normal((128, 16)).astype(np.float32)
    b = rng.standard_normal((n, 16)).astype(np.float32)
    at = torch.from_numpy(a).to(torch.bfloat16).cuda()
    bt = torch.from_numpy(b).to(torch.bfloat16).cuda()
    d = torch.zeros((128, n), dtype=torch.float32, device="cuda")
    mf.diag_umma(at, bt, d, n, a_in_tmem)
    torch.cuda.synchronize()
    ref = at.double().cpu().numpy() @ bt.double().cpu().numpy().T
    np.testing.assert_allclose(d.cpu().numpy(), ref, rtol=1e-5, atol=1e-5)
