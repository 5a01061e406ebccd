"""Backward pass (dq, dk, dv) against the float64 oracle's vector-Jacobian product."""
import numpy as np
import pytest

from gpu_util import TOL_GRAD, TOL_ROW_SHARP_GRAD, rel, require_cuda, row_errors, to_dev

pytestmark = pytest.mark.gpu


def run(q, k, v, do, M, S, T):
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    tq, tk, tv, tdo = (to_dev(x, dev, torch.bfloat16) for x in (q, k, v, do))
    o, lse, _ = bla.bla_forward_chunked(tq, tk, tv, M, S, T)
    dq, dk, dv = bla.bla_backward(tq, tk, tv, o, tdo, lse, M, S, T)
    bla.bla_device_error()
    return [x.float().cpu().numpy() for x in (dq, dk, dv)]


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (1, 2, 300, 64, 32, 32, 256.0),       # 2M = 64, S = 32, ragged
    (2, 1, 260, 128, 64, 64, 1024.0),     # 2M = 128
    (1, 1, 400, 128, 128, 128, 4096.0),   # 2M = 256 (two row tiles for the state GEMMs)
    (1, 2, 128, 64, 64, 64, 200.0),       # exactly one chunk
    (1, 1, 5, 64, 32, 32, 100.0),         # five tokens
])
def test_gradients_against_oracle(orc, B, H, L, d, M, S, T):
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + d)
    do = make_dout(B, H, L, d, dtype="bf16", seed=L + d)
    got = run(q, k, v, do, M, S, T)
    ref = orc.backward(q, k, v, do, M, S, T)
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        assert rel(a, b) <= TOL_GRAD, (name, rel(a, b))


def test_gradients_sharp_softmax(orc):
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    q, k, v = make_qkv(1, 1, 500, 128, dtype="bf16", seed=77, sharp=True)
    do = make_dout(1, 1, 500, 128, dtype="bf16", seed=77)
    got = run(q, k, v, do, 64, 64, 512.0)
    ref = orc.backward(q, k, v, do, 64, 64, 512.0)
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        assert rel(a, b) <= TOL_GRAD, (name, rel(a, b))


def test_lm_layer_workload_gradients_sharp_sampled_heads(orc):
    """The LM-layer shape (B=8, H=8, L=4096, d=128, M=64, S=64, T=1024) with sharp q, k ~ N(0,1):
    the full-size backward recomputes p from an lse taken at |s| up to ~30; every gradient of three
    sampled (batch, head) pairs against the oracle, pooled and per row."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, workload_inputs
    w = WORKLOADS["fwdbwd_bf16_lm"]
    x = workload_inputs(w, seed=0, sharp=True)
    got = run(x["q"], x["k"], x["v"], x["dout"], w.M, w.S, w.T)
    for b, h in ((0, 0), (3, 5), (7, 7)):
        sl = (slice(b, b + 1), slice(h, h + 1))
        ref = orc.backward(x["q"][sl], x["k"][sl], x["v"][sl], x["dout"][sl], w.M, w.S, w.T)
        for name, a, r in zip(("dq", "dk", "dv"), got, ref):
            pooled, worst = row_errors(a[sl], r)
            assert pooled <= TOL_GRAD, (name, b, h, pooled)
            assert worst <= TOL_ROW_SHARP_GRAD, (name, b, h, worst)


def test_lm_layer_workload_gradients_sampled_heads(orc):
    """B=8, H=8, L=4096, d=128, M=64, S=64, T=1024, dO ~ N(0,1): the full-size backward on the GPU;
    every gradient of three sampled (batch, head) pairs against the oracle (heads are independent)."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, workload_inputs
    w = WORKLOADS["fwdbwd_bf16_lm"]
    x = workload_inputs(w, seed=0)
    got = run(x["q"], x["k"], x["v"], x["dout"], w.M, w.S, w.T)
    for b, h in ((0, 0), (3, 5), (7, 7)):
        sl = (slice(b, b + 1), slice(h, h + 1))
        ref = orc.backward(x["q"][sl], x["k"][sl], x["v"][sl], x["dout"][sl], w.M, w.S, w.T)
        for name, a, r in zip(("dq", "dk", "dv"), got, ref):
            pooled, worst = row_errors(a[sl], r)
            assert pooled <= TOL_GRAD, (name, b, h, pooled)
            assert worst <= TOL_GRAD, (name, b, h, worst)
