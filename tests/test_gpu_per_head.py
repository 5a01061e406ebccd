"""Per-head periods (Alg. 1 and Alg. 3 take T in R^H): the fp32 forward, the bf16 tensor-core forward
(device and host buffers) and backward, both decode entry points and the state-decay entry points,
against the oracle run at each head's own period."""
import numpy as np
import pytest

from gpu_util import TOL_BF16, TOL_F32, TOL_GRAD, lse_bound, rel, require_cuda, row_errors, to_dev

pytestmark = pytest.mark.gpu

TS = [7.0, 16.0, 40.0]   # one head at T = 2M-1 = S (M = 4, S = 7), two blurry ones


@pytest.mark.parametrize("phase_mode", ["lag", "absolute"])
def test_f32_forward(orc, phase_mode):
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    B, H, L, d, M, S = 2, 3, 150, 32, 4, 7
    q, k, v = make_qkv(B, H, L, d, dtype="f32", seed=5)
    o, lse, st = bla.bla_forward_chunked(*(to_dev(x, dev, torch.float32) for x in (q, k, v)), M, S, TS, chunk=32,
                                         want_state=True, phase_mode=phase_mode)
    bla.bla_device_error()
    form = "naive" if phase_mode == "lag" else "absolute"
    ref = orc.forward(q, k, v, M, S, TS, form=form)
    assert rel(o.cpu().numpy(), ref["o"]) <= TOL_F32
    assert np.abs(lse.cpu().numpy() - ref["lse"]).max() <= 1e-4
    st_ref = orc.forward(q, k, v, M, S, TS, form="modes", return_state=True)["state"]
    assert rel(st.cpu().numpy(), st_ref) <= TOL_F32


@pytest.mark.parametrize("dtype,phase_mode", [("f32", "lag"), ("bf16", "lag"), ("bf16", "absolute")])
def test_decode_from_zero_state(orc, dtype, phase_mode):
    """Decode steps from the zero state at pos = 0, 1, ... reproduce the forward over the sequence."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    B, H, L, d, M, S = 2, 3, 40, 64, 4, 7
    q, k, v = make_qkv(B, H, L, d, dtype=dtype, seed=9)
    st = torch.zeros((B, H, 2, M, 2, d), dtype=torch.float32, device=dev)
    outs = []
    for t in range(L):
        o = bla.bla_decode_step(to_dev(q[:, :, t], dev, tdt), to_dev(k[:, :, t], dev, tdt), to_dev(v[:, :, t], dev, tdt),
                                st, t, M, S, TS, phase_mode=phase_mode)
        outs.append(o.float().cpu().numpy())
    bla.bla_device_error()
    form = "naive" if phase_mode == "lag" else "absolute"
    ref = orc.forward(q, k, v, M, S, TS, form=form)
    assert rel(np.stack(outs, 2), ref["o"]) <= (TOL_F32 if dtype == "f32" else TOL_BF16)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_decay_forward_and_decode(orc, dtype):
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    tol = TOL_F32 if dtype == "f32" else TOL_BF16
    B, H, L, L1, d, M, S = 2, 3, 120, 90, 64, 4, 7
    q, k, v = make_qkv(B, H, L, d, dtype=dtype, seed=13)
    full = orc.forward_decay(q, k, v, M, S, TS, return_state=True)
    o1, _, st = bla.bla_decay_forward(*(to_dev(x[:, :, :L1], dev, tdt) for x in (q, k, v)), M, S, TS, want_state=True)
    outs = [o1.float().cpu().numpy()]
    for t in range(L1, L):
        o = bla.bla_decay_decode_step(to_dev(q[:, :, t], dev, tdt), to_dev(k[:, :, t], dev, tdt),
                                      to_dev(v[:, :, t], dev, tdt), st, t, M, S, TS)
        outs.append(o.float().cpu().numpy()[:, :, None])
    bla.bla_device_error()
    assert rel(np.concatenate(outs, 2), full["o"]) <= tol
    assert rel(st.cpu().numpy(), full["state"]) <= tol


def test_shared_period_unchanged(orc):
    """Equal per-head periods give the shared-period result."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    q, k, v = (to_dev(x, dev, torch.float32) for x in make_qkv(1, 3, 70, 32, dtype="f32", seed=2))
    a = bla.bla_forward_chunked(q, k, v, 4, 7, [16.0] * 3, chunk=16)[0]
    b = bla.bla_forward_chunked(q, k, v, 4, 7, 16.0, chunk=16)[0]
    bla.bla_device_error()
    assert rel(a.cpu().numpy(), b.cpu().numpy()) <= 1e-6


def test_decay_backward(orc):
    """The decayed VJP with one period per head against the oracle's per-head VJP."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    dev = require_cuda()
    B, H, L, d, M, S = 1, 3, 60, 32, 4, 7
    q, k, v = make_qkv(B, H, L, d, dtype="f32", seed=17)
    do = make_dout(B, H, L, d, dtype="f32", seed=17)
    tq, tk, tv, tdo = (to_dev(x, dev, torch.float32) for x in (q, k, v, do))
    o, lse, _ = bla.bla_decay_forward(tq, tk, tv, M, S, TS)
    got = bla.bla_decay_backward(tq, tk, tv, o, tdo, lse, M, S, TS)
    bla.bla_device_error()
    ref = orc.backward_decay(q, k, v, do, M, S, TS)
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        assert rel(a.cpu().numpy(), b) <= 1e-4, (name, rel(a.cpu().numpy(), b))


@pytest.mark.parametrize("B,H,L,d,M,S,TH,phase_mode", [
    # 2M = 64: an integer, a clamped (T < 2M-1) and a fractional period (fp64 phases)
    (2, 3, 700, 64, 32, 32, [256.0, 40.0, 1000.5], "lag"),
    (2, 3, 700, 64, 32, 32, [256.0, 40.0, 1000.5], "absolute"),
    # 2M = 256 (two mode halves), one-chunk segments: per-head FSEG tables in the prepass and scan
    (1, 2, 3000, 128, 128, 128, [4096.0, 1500.0], "lag"),
    # 2M = 128 with S = 64, ragged tail, three heads of one batch element each
    (3, 2, 333, 128, 64, 64, [1024.0, 200.0], "lag"),
])
def test_bf16_forward(orc, B, H, L, d, M, S, TH, phase_mode):
    """The tensor-core passes with one EB, PHI, FSEG and slot-lag table per head, against the oracle."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + H)
    o, lse, st = bla.bla_forward_chunked(*(to_dev(x, dev, torch.bfloat16) for x in (q, k, v)), M, S, TH,
                                         want_state=True, phase_mode=phase_mode)
    bla.bla_device_error()
    form = "modes" if phase_mode == "lag" else "absolute"
    ref = orc.forward(q, k, v, M, S, TH, form=form)
    pooled, worst = row_errors(o.float().cpu().numpy(), ref["o"])
    assert pooled <= TOL_BF16 and worst <= TOL_BF16, (pooled, worst)
    lse = lse.cpu().numpy()
    assert np.all(np.abs(lse - ref["lse"]) <= lse_bound(ref["lse"])), np.abs(lse - ref["lse"]).max()
    st_ref = orc.forward(q, k, v, M, S, TH, form="modes", return_state=True)["state"]
    assert rel(st.cpu().numpy(), st_ref) <= TOL_BF16
    # each head alone at its own scalar period gives the same result (tables indexed per head)
    for h in range(H):
        oh = bla.bla_forward_chunked(*(to_dev(x[:, h:h + 1], dev, torch.bfloat16) for x in (q, k, v)), M, S, TH[h],
                                     phase_mode=phase_mode)[0]
        assert rel(oh.float().cpu().numpy(), o[:, h:h + 1].float().cpu().numpy()) <= 1e-2


def test_bf16_host_buffer_forward_groups_cross_batches(orc):
    """B=3, H=5, L=12000, d=128 (184 MB: two pipelined head groups that split a batch element) with one
    period per head: equals the device-buffer forward, whose heads the oracle checks above."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    TH = [1024.0, 300.0, 700.0, 2048.0, 129.0]
    q, k, v = make_qkv(3, 5, 12000, 128, dtype="bf16", seed=31)
    hq, hk, hv = (torch.from_numpy(x).to(torch.bfloat16).pin_memory() for x in (q, k, v))
    o_host = bla.bla_forward_chunked_host(hq, hk, hv, 64, 64, TH)
    torch.cuda.synchronize()
    bla.bla_device_error()
    o_dev = bla.bla_forward_chunked(hq.to(dev), hk.to(dev), hv.to(dev), 64, 64, TH)[0].cpu()
    assert rel(o_host.float().numpy(), o_dev.float().numpy()) <= 1e-2
    want = np.zeros(12000, bool)
    want[::101] = True
    want[-2:] = True
    ref = orc.forward(q[1:2], k[1:2], v[1:2], 64, 64, TH, form="modes", want=want)
    got = o_host.float().numpy()[1:2]
    assert rel(got[:, :, want], ref["o"][:, :, want]) <= TOL_BF16


def test_noalloc_decode_matches_workspace_decode():
    """The no-alloc decode builds every head's tables in its fixed scratch and matches bla_decode_step."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_decode_step, make_state
    dev = require_cuda()
    B, H, d, M, S = 4, 3, 128, 32, 32
    TH = [64.0, 256.0, 1000.5]
    st0 = torch.from_numpy(make_state(B, H, M, d, std=0.1, seed=7)).to(dev)
    sa, sb = st0.clone(), st0.clone()
    for step in range(3):
        q, k, v = (to_dev(x, dev, torch.bfloat16) for x in make_decode_step(step, B, H, d, "bf16", seed=7))
        oa = bla.bla_decode_step(q, k, v, sa, 1100 + step, M, S, TH)
        ob = bla.bla_decode_step_noalloc(q, k, v, sb, 1100 + step, M, S, TH)
        torch.cuda.synchronize()
        assert rel(ob.float().cpu().numpy(), oa.float().cpu().numpy()) <= 1e-6
    assert rel(sb.cpu().numpy(), sa.cpu().numpy()) <= 1e-6
    bla.bla_device_error()


@pytest.mark.parametrize("phase_mode", ["lag", "absolute"])
def test_bf16_backward(orc, phase_mode):
    """The bf16 backward with one period per head (the heads run one at a time, each at its period),
    against the oracle's VJP; rows compared within their head."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    dev = require_cuda()
    B, H, L, d, M, S = 2, 3, 300, 64, 32, 32
    TH = [256.0, 40.0, 1000.5]
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=51)
    do = make_dout(B, H, L, d, dtype="bf16", seed=51)
    tq, tk, tv, tdo = (to_dev(x, dev, torch.bfloat16) for x in (q, k, v, do))
    o, lse, _ = bla.bla_forward_chunked(tq, tk, tv, M, S, TH, phase_mode=phase_mode)
    got = bla.bla_backward(tq, tk, tv, o, tdo, lse, M, S, TH, phase_mode=phase_mode)
    bla.bla_device_error()
    ref = orc.backward(q, k, v, do, M, S, TH, form="parallel" if phase_mode == "lag" else "absolute")
    for name, a, r in zip(("dq", "dk", "dv"), got, ref):
        a = a.float().cpu().numpy()
        assert rel(a, r) <= TOL_GRAD, (name, rel(a, r))
        for b in range(B):
            for h in range(H):
                assert row_errors(a[b, h], r[b, h])[1] <= TOL_GRAD, (name, b, h)
