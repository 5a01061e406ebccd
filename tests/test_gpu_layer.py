"""A BLA layer in an LM block (RegBench-sized: d_model 128, 4 heads, M = 16, S = 2M-1 = 31,
T = 2(2M-1)): projections by cuBLAS, token mixing by the library's fp32 path, against the same
composition in float64 with the oracle."""
import numpy as np
import pytest

from gpu_util import TOL_F32, rel, require_cuda

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("phase_mode,form", [("lag", "modes"), ("absolute", "absolute")])
def test_lm_block_layer(orc, phase_mode, form):
    import torch
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_block_inputs
    from paper_2606_09862_gb300.layer import bla_block_forward
    dev = require_cuda()
    w = WORKLOADS["lm_block_f32"]
    B, L, dm = 4, w.L, w.H * w.d
    x, ws = make_block_inputs(B, L, dm, seed=2)
    torch.backends.cuda.matmul.allow_tf32 = False
    t = lambda a: torch.from_numpy(a).to(dev)
    y = bla_block_forward(t(x), *(t(a) for a in ws), w.H, w.M, w.S, w.T, phase_mode=phase_mode)
    torch.cuda.synchronize()
    xd = x.astype(np.float64)
    wq, wk, wv, wo = (a.astype(np.float64) for a in ws)
    heads = lambda a: a.reshape(B, L, w.H, w.d).transpose(0, 2, 1, 3)
    o = orc.forward(heads(xd @ wq), heads(xd @ wk), heads(xd @ wv), w.M, w.S, w.T, form=form)["o"]
    ref = o.transpose(0, 2, 1, 3).reshape(B, L, dm) @ wo
    assert rel(y.cpu().numpy(), ref) <= TOL_F32, rel(y.cpu().numpy(), ref)
