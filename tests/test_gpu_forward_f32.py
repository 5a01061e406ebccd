"""fp32 chunked forward (CUDA cores) against the float64 oracle."""
import numpy as np
import pytest

from gpu_util import TOL_F32, rel, require_cuda, to_dev

pytestmark = pytest.mark.gpu


def run(q, k, v, M, S, T, chunk=0, omega=0.0, want_state=True):
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    o, lse, st = bla.bla_forward_chunked(to_dev(q, dev, torch.float32), to_dev(k, dev, torch.float32),
                                         to_dev(v, dev, torch.float32), M, S, T, omega=omega, chunk=chunk,
                                         want_state=want_state)
    torch.cuda.synchronize()
    return o.cpu().numpy(), lse.cpu().numpy(), (st.cpu().numpy() if st is not None else None)


def test_config_fwd_f32_small(orc):
    """B=1, H=2, L=256, d=32, M=16, S=16, T=64, chunk 64; N(0,1)/sqrt(d); seed 0."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, workload_inputs
    w = WORKLOADS["fwd_f32_small"]
    x = workload_inputs(w, seed=0)
    o, lse, st = run(x["q"], x["k"], x["v"], w.M, w.S, w.T, chunk=w.chunk)
    ref = orc.forward(x["q"], x["k"], x["v"], w.M, w.S, w.T, return_state=True)
    assert rel(o, ref["o"]) <= TOL_F32
    assert np.abs(lse - ref["lse"]).max() <= 1e-4
    assert rel(st, ref["state"]) <= TOL_F32


def test_sharp_softmax(orc):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 2, 256, 32, dtype="f32", seed=5, sharp=True)
    o, lse, st = run(q, k, v, 16, 16, 64.0, chunk=64)
    ref = orc.forward(q, k, v, 16, 16, 64.0, return_state=True)
    assert rel(o, ref["o"]) <= TOL_F32
    assert rel(st, ref["state"]) <= TOL_F32


@pytest.mark.parametrize("L,chunk", [(1, 64), (2, 64), (63, 64), (65, 64), (130, 64), (100, 1), (100, 7),
                                     (100, 100), (257, 128)])
def test_ragged_and_chunk_independence(orc, L, chunk):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(2, 1, L, 16, dtype="f32", seed=L)
    o, lse, st = run(q, k, v, 6, 5, 23.0, chunk=chunk)
    ref = orc.forward(q, k, v, 6, 5, 23.0, return_state=True)
    assert rel(o, ref["o"]) <= TOL_F32
    assert np.abs(lse - ref["lse"]).max() <= 1e-4
    assert rel(st, ref["state"]) <= TOL_F32


@pytest.mark.parametrize("M,S,T,omega", [(1, 1, 5.0, 0.0), (4, 7, 7.0, 0.0), (5, 3, 4.0, 0.0),
                                         (3, 11, 11.0, 0.0), (4, 4, 16.0, 0.3)])
def test_degenerate_and_paper_cases(orc, M, S, T, omega):
    """M = 1 (a running sum), full resolution T = S = 2M-1, clamped T < 2M-1, S = T, explicit omega."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 3, 50, 8, dtype="f32", seed=M * 100 + S)
    o, lse, st = run(q, k, v, M, S, T, chunk=16, omega=omega)
    ref = orc.forward(q, k, v, M, S, T, omega=omega, return_state=True)
    assert rel(o, ref["o"]) <= TOL_F32
    assert rel(st, ref["state"]) <= TOL_F32


def test_empty_sequence():
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    z = torch.zeros((1, 2, 0, 8), device=dev)
    o, lse, st = bla.bla_forward_chunked(z, z, z, 3, 3, 5.0, want_state=True)
    torch.cuda.synchronize()
    assert o.shape == (1, 2, 0, 8)
    assert float(st.abs().max()) == 0.0


@pytest.mark.parametrize("L", [1, 2, 63, 65])
@pytest.mark.parametrize("M,S,T", [(1, 1, 5.0), (4, 7, 7.0), (3, 5, 12.0)])
def test_tiny_shapes_every_output_written(orc, L, M, S, T):
    """Tiny shapes around the chunk boundary (C = 64): L in {1, 2, C-1, C+1}, down to one mode and
    one slot; o is prefilled with NaN so that an element the kernel skips fails the test."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    q, k, v = make_qkv(2, 1, L, 8, dtype="f32", seed=L + 10 * M)
    out = torch.full((2, 1, L, 8), float("nan"), device=dev)
    o, lse, st = bla.bla_forward_chunked(to_dev(q, dev, torch.float32), to_dev(k, dev, torch.float32),
                                         to_dev(v, dev, torch.float32), M, S, T, chunk=64, out=out,
                                         want_state=True)
    torch.cuda.synchronize()
    assert torch.isfinite(o).all() and torch.isfinite(lse).all()
    ref = orc.forward(q, k, v, M, S, T, form="naive", return_state=True)
    assert rel(o.cpu().numpy(), ref["o"]) <= TOL_F32
    assert rel(st.cpu().numpy(), ref["state"]) <= TOL_F32
