"""Helpers of the GPU tests: layout conversion and one call through the C ABI."""
import numpy as np


def from_planar(xp, C):
    from paper_2107_06960_gb300 import from_planar as fp
    return fp(xp, C)


def run_plan(mf, layers, params, x, cut, grids, dtype, plan_kwargs=None, repeat=1):
    """Run one plan on x [B][H][W][C]; returns (cut tensor NHWC or None, output NHWC) as float32."""
    import torch
    B, H, W, C = x.shape
    net = mf.Net(layers, H, W, C)
    net.set_params(params)
    plan = mf.Plan(net, cut, grids, batch=B, dtype=dtype, **(plan_kwargs or {}))
    tdt = torch.bfloat16 if dtype == mf.BF16 else torch.float32
    xin = torch.from_numpy(np.ascontiguousarray(x)).to(tdt).cuda()  # NHWC, as the image comes
    n = len(layers)
    sh = net.shape(n - 1)
    out = torch.full((B, sh[3], sh[4], sh[5]), float("nan"), dtype=tdt, device="cuda")
    cut_out = None
    cut_c = None
    if cut is not None:  # the cut tensor is group 1's output
        sc = net.shape((cut[0] if isinstance(cut, (list, tuple)) else cut) - 1)
        cut_c = sc[5]
        cut_out = torch.full((B, (sc[5] + 7) // 8, sc[3], sc[4], 8), float("nan"), dtype=tdt, device="cuda")
    for _ in range(repeat):
        plan.run_debug(xin, cut_out, out)
    plan.sync_status(like=xin)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    c = from_planar(cut_out.float().cpu().numpy(), cut_c) if cut_out is not None else None
    plan.close()
    return c, o


def rel_err(got, ref):
    """max |got - ref| / max |ref| (the tolerance norm of the parity tests)."""
    den = float(np.abs(ref).max())
    return float(np.abs(got - ref).max()) / (den if den > 0 else 1.0)
