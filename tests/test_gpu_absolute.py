"""The absolute-phase form (Alg. 1, Sec. 3.2; phase_mode "absolute") on every path against the
oracle's Alg. 1 forward and its VJP.

The mode state is the same object in both forms (the running sums of Eq. recurrence), so the
final states are checked against the oracle's lag-form recurrence.
"""
import numpy as np
import pytest

from gpu_util import (TOL_BF16, TOL_F32, TOL_GRAD, TOL_ROW_BF16, TOL_ROW_SHARP, lse_bound, rel, require_cuda,
                      row_errors, to_dev)

pytestmark = pytest.mark.gpu

ABS = "absolute"


def fwd(q, k, v, M, S, T, dtype, chunk=0, phase_mode=ABS):
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    o, lse, st = bla.bla_forward_chunked(to_dev(q, dev, tdt), to_dev(k, dev, tdt), to_dev(v, dev, tdt), M, S, T,
                                         chunk=chunk, want_state=True, phase_mode=phase_mode)
    bla.bla_device_error()
    return o.float().cpu().numpy(), lse.cpu().numpy(), st.cpu().numpy()


@pytest.mark.parametrize("L,chunk", [(256, 64), (203, 48), (1, 64)])
def test_f32_against_alg1(orc, L, chunk):
    """B=1, H=2, d=32, M=16, S=16, T=64 (the small fp32 workload's shape), ragged and 1-token cases."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 2, L, 32, dtype="f32", seed=L)
    o, lse, st = fwd(q, k, v, 16, 16, 64.0, "f32", chunk=chunk)
    ref = orc.forward(q, k, v, 16, 16, 64.0, form="absolute")
    assert rel(o, ref["o"]) <= TOL_F32, rel(o, ref["o"])
    assert np.abs(lse - ref["lse"]).max() <= 1e-4
    st_ref = orc.forward(q, k, v, 16, 16, 64.0, form="modes", return_state=True)["state"]
    assert rel(st, st_ref) <= TOL_F32


def test_f32_forms_coincide_at_full_resolution():
    """T = S = 2M-1: the two forms give the same outputs (Sec. 3.2's equivalence), and differ for
    T > 2M-1."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 2, 90, 16, dtype="f32", seed=4)
    a = fwd(q, k, v, 4, 7, 7.0, "f32", chunk=32)[0]
    b = fwd(q, k, v, 4, 7, 7.0, "f32", chunk=32, phase_mode="lag")[0]
    assert rel(a, b) <= TOL_F32
    a = fwd(q, k, v, 4, 7, 16.0, "f32", chunk=32)[0]
    b = fwd(q, k, v, 4, 7, 16.0, "f32", chunk=32, phase_mode="lag")[0]
    assert rel(a, b) > 1e-2


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (2, 2, 300, 64, 32, 32, 256.0),      # 2M = 64, ragged tail
    (1, 2, 1000, 128, 64, 64, 1024.0),   # 2M = 128, many segments (prepass + scan)
    (1, 1, 777, 128, 128, 128, 4096.0),  # 2M = 256 (two mode halves), multi-segment
    (3, 1, 129, 64, 128, 32, 512.0),     # 2M = 256 with d = 64, S = 32
    (2, 1, 1, 64, 32, 64, 100.0),        # a single token
])
def test_bf16_against_alg1(orc, B, H, L, d, M, S, T):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + M + 1)
    o, lse, st = fwd(q, k, v, M, S, T, "bf16")
    ref = orc.forward(q, k, v, M, S, T, form="absolute")
    assert rel(o, ref["o"]) <= TOL_BF16, rel(o, ref["o"])
    assert np.abs(lse - ref["lse"]).max() <= 5e-2
    st_ref = orc.forward(q, k, v, M, S, T, form="modes", return_state=True)["state"]
    assert rel(st, st_ref) <= TOL_BF16


def test_bf16_long_multisegment(orc):
    """B=1, H=4, L=16384, d=128, M=128, S=128, T=4096: nine segments per head, sampled tokens."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 4, 16384, 128, dtype="bf16", seed=5)
    o, lse, st = fwd(q, k, v, 128, 128, 4096.0, "bf16")
    ref = orc.forward(q, k, v, 128, 128, 4096.0, form="absolute")
    want = np.zeros(16384, bool)
    want[::37] = True
    want[127::128] = True
    want[-3:] = True
    pooled, worst = row_errors(o[:, :, want], ref["o"][:, :, want])
    assert pooled <= TOL_BF16, pooled
    assert worst <= TOL_ROW_BF16, worst
    assert np.abs(lse[:, :, want] - ref["lse"][:, :, want]).max() <= 5e-2


def test_bf16_sharp_softmax(orc):
    """q, k ~ N(0,1): o pooled and per row, and lse per token, against Alg. 1."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 2, 2000, 128, dtype="bf16", seed=8, sharp=True)
    o, lse, _ = fwd(q, k, v, 128, 128, 4096.0, "bf16")
    ref = orc.forward(q, k, v, 128, 128, 4096.0, form="absolute")
    pooled, worst = row_errors(o, ref["o"])
    assert pooled <= TOL_BF16, pooled
    assert worst <= TOL_ROW_SHARP, worst
    assert np.all(np.abs(lse - ref["lse"]) <= lse_bound(ref["lse"])), np.abs(lse - ref["lse"]).max()


@pytest.mark.parametrize("dtype,noalloc", [("f32", False), ("bf16", False), ("bf16", True)])
def test_decode_continues_prefill(orc, dtype, noalloc):
    """Prefill of L1 tokens, then decode steps at pos = L1.. in the absolute form, equals Alg. 1 over
    the whole sequence."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    if dtype == "f32":
        B, H, L, d, M, S, T, L1 = 1, 2, 60, 64, 5, 9, 20.0, 37
    else:
        B, H, L, d, M, S, T, L1 = 2, 2, 330, 64, 32, 32, 256.0, 300
    q, k, v = make_qkv(B, H, L, d, dtype=dtype, seed=12)
    _, _, st = bla.bla_forward_chunked(to_dev(q[:, :, :L1], dev, tdt), to_dev(k[:, :, :L1], dev, tdt),
                                       to_dev(v[:, :, :L1], dev, tdt), M, S, T, chunk=16 if dtype == "f32" else 0,
                                       want_state=True, phase_mode=ABS)
    step = bla.bla_decode_step_noalloc if noalloc else bla.bla_decode_step
    outs = []
    for t in range(L1, L):
        o = step(to_dev(q[:, :, t], dev, tdt), to_dev(k[:, :, t], dev, tdt), to_dev(v[:, :, t], dev, tdt), st, t,
                 M, S, T, phase_mode=ABS)
        outs.append(o.float().cpu().numpy())
    bla.bla_device_error()
    ref = orc.forward(q, k, v, M, S, T, form="absolute")
    tol = TOL_F32 if dtype == "f32" else TOL_BF16
    assert rel(np.stack(outs, 2), ref["o"][:, :, L1:]) <= tol
    st_ref = orc.forward(q, k, v, M, S, T, form="modes", return_state=True)["state"]
    assert rel(st.cpu().numpy(), st_ref) <= tol


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (1, 2, 300, 64, 32, 32, 256.0),       # 2M = 64, ragged
    (2, 1, 260, 128, 64, 64, 1024.0),     # 2M = 128
    (1, 1, 400, 128, 128, 128, 4096.0),   # 2M = 256
])
def test_backward_against_alg1_vjp(orc, B, H, L, d, M, S, T):
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    dev = require_cuda()
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + 3)
    do = make_dout(B, H, L, d, dtype="bf16", seed=L + 3)
    tq, tk, tv, tdo = (to_dev(x, dev, torch.bfloat16) for x in (q, k, v, do))
    o, lse, _ = bla.bla_forward_chunked(tq, tk, tv, M, S, T, phase_mode=ABS)
    got = bla.bla_backward(tq, tk, tv, o, tdo, lse, M, S, T, phase_mode=ABS)
    bla.bla_device_error()
    ref = orc.backward(q, k, v, do, M, S, T, form="absolute")
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        a = a.float().cpu().numpy()
        assert rel(a, b) <= TOL_GRAD, (name, rel(a, b))
