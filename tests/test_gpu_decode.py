"""Single-token decode against the oracle recurrence."""
import numpy as np
import pytest

from gpu_util import TOL_BF16, TOL_F32, TOL_ROW_BF16, rel, require_cuda, row_errors, to_dev

pytestmark = pytest.mark.gpu


def test_decode_small_every_head(orc):
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_decode_step, make_state
    dev = require_cuda()
    B, H, d, M, S, T, pos0, steps = 3, 2, 32, 8, 6, 30.0, 5, 40
    st0 = make_state(B, H, M, d, std=0.1, seed=1)
    tst = torch.from_numpy(st0).to(dev)
    qs, ks, vs, outs = [], [], [], []
    for s in range(steps):
        q, k, v = make_decode_step(s, B, H, d, dtype="f32", seed=1)
        qs.append(q); ks.append(k); vs.append(v)
        o = bla.bla_decode_step(to_dev(q, dev, torch.float32), to_dev(k, dev, torch.float32),
                                to_dev(v, dev, torch.float32), tst, pos0 + s, M, S, T)
        outs.append(o.cpu().numpy())
    stk = lambda xs: np.stack(xs, axis=2)       # [B,H,steps,d]
    ref = orc.forward(stk(qs), stk(ks), stk(vs), M, S, T, state=st0, pos0=pos0, return_state=True)
    assert rel(stk(outs), ref["o"]) <= TOL_F32
    assert rel(tst.cpu().numpy(), ref["state"]) <= TOL_F32


def test_decode_continues_prefill(orc):
    """Prefill of L1 tokens (state_out) then decode steps at pos = L1.. equals one pass (Eq. recurrence)."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    B, H, L, d, M, S, T, L1 = 1, 2, 40, 64, 5, 9, 20.0, 25
    q, k, v = make_qkv(B, H, L, d, dtype="f32", seed=7)
    _, _, st = bla.bla_forward_chunked(to_dev(q[:, :, :L1], dev, torch.float32),
                                       to_dev(k[:, :, :L1], dev, torch.float32),
                                       to_dev(v[:, :, :L1], dev, torch.float32), M, S, T, chunk=8, want_state=True)
    outs = []
    for t in range(L1, L):
        o = bla.bla_decode_step(to_dev(q[:, :, t], dev, torch.float32), to_dev(k[:, :, t], dev, torch.float32),
                                to_dev(v[:, :, t], dev, torch.float32), st, t, M, S, T)
        outs.append(o.cpu().numpy())
    ref = orc.forward(q, k, v, M, S, T, return_state=True)
    assert rel(np.stack(outs, 2), ref["o"][:, :, L1:]) <= TOL_F32
    assert rel(st.cpu().numpy(), ref["state"]) <= TOL_F32


def test_decode_masking_from_sequence_start(orc):
    """From the zero state at pos 0 the slot mask hides slots with D_j > pos (Eq. output)."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    B, H, L, d, M, S, T = 2, 1, 12, 128, 4, 7, 14.0
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=9, sharp=True)
    st = torch.zeros((B, H, 2, M, 2, d), device=dev)
    outs = []
    for t in range(L):
        o = bla.bla_decode_step(to_dev(q[:, :, t], dev, torch.bfloat16), to_dev(k[:, :, t], dev, torch.bfloat16),
                                to_dev(v[:, :, t], dev, torch.bfloat16), st, t, M, S, T)
        outs.append(o.float().cpu().numpy())
    ref = orc.forward(q, k, v, M, S, T)
    assert rel(np.stack(outs, 2), ref["o"]) <= TOL_BF16


def test_decode_workload_1024_steps(orc):
    """256 sequences x 16 heads, d=128, M=128, S=128, T=4096, fp32 state ~ N(0, 0.1^2),
    1024 consecutive bf16 steps from pos 4096; every step's output and the final state of
    sampled heads checked against the oracle recurrence."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_decode_step, make_state
    dev = require_cuda()
    w = WORKLOADS["decode_bf16"]
    B, H, d, M, S, T = w.B, w.H, w.d, w.M, w.S, w.T
    st0 = make_state(B, H, M, d, std=w.state_std, seed=0)
    tst = torch.from_numpy(st0).to(dev)
    rng = np.random.default_rng(123)
    heads = [(0, 0), (B - 1, H - 1)] + [(int(rng.integers(B)), int(rng.integers(H))) for _ in range(6)]
    bi = np.array([h[0] for h in heads]); hi = np.array([h[1] for h in heads])
    nsteps = w.decode_steps
    qs = np.zeros((len(heads), 1, nsteps, d), np.float32)
    ks, vs, outs = np.zeros_like(qs), np.zeros_like(qs), np.zeros_like(qs)
    ws = torch.empty(bla.bla_workspace_bytes(bla.make_params(B, H, 1, d, d, M, S, T), bla.BLA_WS_DECODE),
                     dtype=torch.uint8, device=dev)
    for s in range(nsteps):
        q, k, v = make_decode_step(s, B, H, d, dtype="bf16", seed=0)
        o = bla.bla_decode_step(to_dev(q, dev, torch.bfloat16), to_dev(k, dev, torch.bfloat16),
                                to_dev(v, dev, torch.bfloat16), tst, w.decode_pos0 + s, M, S, T, workspace=ws)
        oc = o.float()[torch.from_numpy(bi).to(dev), torch.from_numpy(hi).to(dev)].cpu().numpy()
        qs[:, 0, s], ks[:, 0, s], vs[:, 0, s], outs[:, 0, s] = q[bi, hi], k[bi, hi], v[bi, hi], oc
    bla.bla_device_error()
    ref = orc.forward(qs, ks, vs, M, S, T, state=st0[bi, hi][:, None], pos0=w.decode_pos0, form="modes",
                      return_state=True)
    worst = max(rel(outs[:, 0, s], ref["o"][:, 0, s]) for s in range(nsteps))
    assert worst <= TOL_BF16, worst
    # every (head, step) output row on its own
    pooled, worst_row = row_errors(outs, ref["o"])
    assert pooled <= TOL_BF16 and worst_row <= TOL_ROW_BF16, (pooled, worst_row)
    assert rel(tst.cpu().numpy()[bi, hi], ref["state"][:, 0]) <= TOL_F32
