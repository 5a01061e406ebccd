"""The state decay of Sec. 3.3 (Alg. 1's slot state multiplied by 1 - D_j(t) before each token is
added) on the GPU, through the C ABI, against the oracle's decayed Alg. 1."""
import numpy as np
import pytest

from gpu_util import TOL_BF16, TOL_F32, TOL_GRAD, TOL_ROW_BF16, rel, require_cuda, row_errors, to_dev

pytestmark = pytest.mark.gpu


def gpu_forward(q, k, v, M, S, T, dtype, pos0=0, state=None):
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    st = None if state is None else to_dev(state, dev, torch.float32)
    o, lse, st = bla.bla_decay_forward(to_dev(q, dev, tdt), to_dev(k, dev, tdt), to_dev(v, dev, tdt), M, S, T,
                                       pos0=pos0, state=st, want_state=True)
    bla.bla_device_error()
    return o.float().cpu().numpy(), lse.cpu().numpy(), st.cpu().numpy()


def check(got, ref, tol, lse_tol):
    o, lse, st = got
    assert rel(o, ref["o"]) <= tol, rel(o, ref["o"])
    assert np.abs(lse - ref["lse"]).max() <= lse_tol
    assert rel(st, ref["state"]) <= tol, rel(st, ref["state"])


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (1, 2, 203, 32, 16, 16, 64.0),     # ragged tails of the 32-token score and 16-token value tiles
    (2, 1, 100, 64, 4, 7, 7.0),        # T = S = 2M-1: sliding-window attention over 7 tokens
    (1, 2, 77, 128, 32, 32, 256.0),
    (1, 1, 50, 64, 8, 200, 300.0),     # 25 slot groups, a partial block of slot warps
    (1, 1, 1, 32, 4, 5, 9.0),          # a single token
])
def test_f32_forward(orc, B, H, L, d, M, S, T):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(B, H, L, d, dtype="f32", seed=L + S)
    check(gpu_forward(q, k, v, M, S, T, "f32"), orc.forward_decay(q, k, v, M, S, T, return_state=True),
          TOL_F32, 1e-4)


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (1, 2, 300, 128, 64, 64, 1024.0),   # the LM-layer (M, S, T), shortened
    (2, 2, 257, 64, 32, 32, 256.0),
    (1, 1, 129, 128, 128, 128, 4096.0),
    (1, 1, 64, 128, 8, 256, 512.0),     # S = 256, the largest slot count (1024-thread value blocks)
])
def test_bf16_forward(orc, B, H, L, d, M, S, T):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + M)
    check(gpu_forward(q, k, v, M, S, T, "bf16"), orc.forward_decay(q, k, v, M, S, T, return_state=True),
          TOL_BF16, 5e-2)


@pytest.mark.parametrize("B,H,L,d,M,S,T", [
    (1, 2, 500, 64, 17, 32, 33.0),      # T = 2M-1: the decay factors reach exact zeros
    (16, 10, 130, 64, 32, 32, 256.0),   # 160 heads: one segment per head
    (1, 1, 1000, 128, 64, 64, 1024.0),  # 16 one-chunk segments
    (2, 1, 63, 128, 32, 64, 512.0),     # one ragged chunk
    (1, 1, 1, 64, 8, 32, 64.0),         # a single token: one item, one state update
    (1, 2, 33, 128, 16, 64, 100.0),     # one chunk and one token
    (1, 2, 97, 128, 16, 32, 64.0),      # S = 32 with d = 128
    (2, 1, 161, 64, 32, 64, 300.0),     # S = 64 with d = 64
])
def test_bf16_chunked_forward(orc, B, H, L, d, M, S, T):
    """The chunked tensor-core form (d in {64, 128}, S in {32, 64}): o per row, lse and state."""
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=L + S)
    o, lse, st = gpu_forward(q, k, v, M, S, T, "bf16")
    ref = orc.forward_decay(q, k, v, M, S, T, return_state=True)
    pooled, worst = row_errors(o, ref["o"])
    assert pooled <= TOL_BF16 and worst <= TOL_ROW_BF16, (pooled, worst)
    assert np.abs(lse - ref["lse"]).max() <= 5e-2
    assert rel(st, ref["state"]) <= TOL_BF16, rel(st, ref["state"])


def test_bf16_chunked_continues_from_state(orc):
    """A chunked forward from a random slot state at pos0 = 777 (mid-chunk phases, every slot visible
    from the start) equals the oracle continued from the same state; and a prefill split in two
    calls equals one call."""
    from paper_2606_09862_gb300.inputs import make_qkv, make_slot_state
    B, H, L, d, M, S, T = 2, 2, 300, 64, 16, 32, 100.0
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=19)
    st0 = make_slot_state(B, H, S, d, 0.1, seed=19)
    got = gpu_forward(q, k, v, M, S, T, "bf16", pos0=777, state=st0)
    check(got, orc.forward_decay(q, k, v, M, S, T, state=st0, pos0=777, return_state=True), TOL_BF16, 5e-2)
    full = orc.forward_decay(q, k, v, M, S, T, return_state=True)
    o1, _, st1 = gpu_forward(q[:, :, :130], k[:, :, :130], v[:, :, :130], M, S, T, "bf16")
    o2, _, st2 = gpu_forward(q[:, :, 130:], k[:, :, 130:], v[:, :, 130:], M, S, T, "bf16", pos0=130, state=st1)
    assert rel(np.concatenate([o1, o2], 2), full["o"]) <= TOL_BF16
    assert rel(st2, full["state"]) <= TOL_BF16


def test_bf16_chunked_per_head_periods(orc):
    """Per-head periods on the chunked form: one D_M table and grid per head."""
    from paper_2606_09862_gb300.inputs import make_qkv
    TH = [33.0, 256.0, 1000.5]
    q, k, v = make_qkv(2, 3, 200, 64, dtype="bf16", seed=23)
    check(gpu_forward(q, k, v, 17, 32, TH, "bf16"), orc.forward_decay(q, k, v, 17, 32, TH, return_state=True),
          TOL_BF16, 5e-2)


def test_bf16_sharp_softmax(orc):
    from paper_2606_09862_gb300.inputs import make_qkv
    q, k, v = make_qkv(1, 2, 400, 128, dtype="bf16", seed=3, sharp=True)
    check(gpu_forward(q, k, v, 64, 64, 1024.0, "bf16"),
          orc.forward_decay(q, k, v, 64, 64, 1024.0, return_state=True), TOL_BF16, 5e-2)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_prefill_continue_and_decode(orc, dtype):
    """Prefill of L1 tokens, a second forward from its state at pos0 = L1, and decode steps from
    the prefill's state at pos = L1, L1 + 1, ... all equal one pass over the whole sequence."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    B, H, L, L1, d, M, S, T = 2, 2, 90, 61, 64, 16, 24, 100.0
    q, k, v = make_qkv(B, H, L, d, dtype=dtype, seed=7)
    tol = TOL_F32 if dtype == "f32" else TOL_BF16
    full = orc.forward_decay(q, k, v, M, S, T, return_state=True)
    o1, _, st1 = gpu_forward(q[:, :, :L1], k[:, :, :L1], v[:, :, :L1], M, S, T, dtype)
    o2, _, st2 = gpu_forward(q[:, :, L1:], k[:, :, L1:], v[:, :, L1:], M, S, T, dtype, pos0=L1, state=st1)
    assert rel(np.concatenate([o1, o2], 2), full["o"]) <= tol
    assert rel(st2, full["state"]) <= tol
    st = to_dev(st1, dev, torch.float32)
    outs = []
    for t in range(L1, L):
        o = bla.bla_decay_decode_step(to_dev(q[:, :, t], dev, tdt), to_dev(k[:, :, t], dev, tdt),
                                      to_dev(v[:, :, t], dev, tdt), st, t, M, S, T)
        outs.append(o.float().cpu().numpy())
    bla.bla_device_error()
    assert rel(np.stack(outs, 2), full["o"][:, :, L1:]) <= tol
    assert rel(st.cpu().numpy(), full["state"]) <= tol


def test_swa_limit_decode(orc):
    """Decode at T = S = 2M-1 from a zero state reproduces sliding-window attention (the oracle's
    pinned limit) step by step, including the first 2M-2 steps where slots are still masked."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_qkv
    dev = require_cuda()
    B, H, L, d, M = 1, 3, 20, 32, 4
    q, k, v = make_qkv(B, H, L, d, dtype="f32", seed=11)
    ref = orc.forward_decay(q, k, v, M, 7, 7.0)
    st = torch.zeros((B, H, 2, 7, d), dtype=torch.float32, device=dev)
    outs = [bla.bla_decay_decode_step(to_dev(q[:, :, t], dev, torch.float32), to_dev(k[:, :, t], dev, torch.float32),
                                      to_dev(v[:, :, t], dev, torch.float32), st, t, M, 7, 7.0).cpu().numpy()
            for t in range(L)]
    bla.bla_device_error()
    assert rel(np.stack(outs, 2), ref["o"]) <= TOL_F32


def test_full_size_forward_sampled(orc):
    """The bench's decay workload (B=8, H=8, L=4096, d=128, M=64, S=64, T=1024, bf16) in one call;
    head (0, 0) against the oracle on the same seeded draw, all outputs finite."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_qkv
    dev = require_cuda()
    w = WORKLOADS["decay_bf16_lm"]
    q, k, v = make_qkv(w.B, w.H, w.L, w.d, dtype="bf16", seed=0)
    o, lse, _ = bla.bla_decay_forward(*(to_dev(x, dev, torch.bfloat16) for x in (q, k, v)), w.M, w.S, w.T)
    bla.bla_device_error()
    o = o.float().cpu().numpy()
    assert np.isfinite(o).all() and np.isfinite(lse.cpu().numpy()).all()
    ref = orc.forward_decay(q[:1, :1], k[:1, :1], v[:1, :1], w.M, w.S, w.T)
    pooled, worst = row_errors(o[:1, :1], ref["o"])
    assert pooled <= TOL_BF16, pooled
    assert worst <= TOL_ROW_BF16, worst


def test_full_size_backward_sampled(orc):
    """The bench's decay workload (B=8, H=8, L=4096, d=128, M=64, S=64, T=1024, bf16): the full
    backward in one call (the chunked form); heads (0, 0) and (7, 7) against the oracle's VJP,
    pooled and per row."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_dout, make_qkv
    dev = require_cuda()
    w = WORKLOADS["decay_bf16_lm"]
    q, k, v = make_qkv(w.B, w.H, w.L, w.d, dtype="bf16", seed=0)
    do = make_dout(w.B, w.H, w.L, w.d, dtype="bf16", seed=0)
    tq, tk, tv, tdo = (to_dev(x, dev, torch.bfloat16) for x in (q, k, v, do))
    o, lse, _ = bla.bla_decay_forward(tq, tk, tv, w.M, w.S, w.T)
    got = [x.float().cpu().numpy() for x in bla.bla_decay_backward(tq, tk, tv, o, tdo, lse, w.M, w.S, w.T)]
    bla.bla_device_error()
    for b, h in ((0, 0), (7, 7)):
        sl = (slice(b, b + 1), slice(h, h + 1))
        ref = orc.backward_decay(q[sl], k[sl], v[sl], do[sl], w.M, w.S, w.T)
        for name, a, r in zip(("dq", "dk", "dv"), got, ref):
            pooled, worst = row_errors(a[sl], r)
            assert pooled <= TOL_GRAD and worst <= TOL_GRAD, (name, b, h, pooled, worst)


def test_full_size_decode_sampled(orc):
    """The decay decode workload (B=256, H=16, d=128, M=128, S=128, T=4096, pos = 4096, random slot
    state) in one call; three heads against the oracle's one-token forward from the same state."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_decode_step, make_slot_state
    dev = require_cuda()
    w = WORKLOADS["decay_decode_bf16"]
    q, k, v = make_decode_step(0, w.B, w.H, w.d, "bf16", seed=0)
    st0 = make_slot_state(w.B, w.H, w.S, w.d, w.state_std, seed=0)
    st = torch.from_numpy(st0).to(dev)
    o = bla.bla_decay_decode_step(*(to_dev(x, dev, torch.bfloat16) for x in (q, k, v)), st, w.decode_pos0,
                                  w.M, w.S, w.T)
    bla.bla_device_error()
    o = o.float().cpu().numpy()
    stn = st.cpu().numpy()
    assert np.isfinite(o).all()
    for b, h in ((0, 0), (17, 5), (255, 15)):
        ref = orc.forward_decay(q[b:b + 1, h:h + 1, None], k[b:b + 1, h:h + 1, None], v[b:b + 1, h:h + 1, None],
                                w.M, w.S, w.T, state=st0[b:b + 1, h:h + 1], pos0=w.decode_pos0, return_state=True)
        assert rel(o[b, h], ref["o"][0, 0, 0]) <= TOL_BF16
        assert rel(stn[b, h], ref["state"][0, 0]) <= TOL_F32


def test_lag_form_rejected():
    """The decay is defined on the absolute form's slots; the lag form is refused before any launch."""
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    x = torch.zeros((1, 1, 8, 32), dtype=torch.float32, device=dev)
    with pytest.raises(bla.BlaError) as e:
        bla.bla_decay_forward(x, x, x, 4, 4, 16.0, phase_mode="lag")
    assert e.value.status == bla.BLA_ERR_UNSUPPORTED


@pytest.mark.parametrize("dtype,B,H,L,d,M,S,T,pos0", [
    ("f32", 1, 2, 70, 32, 8, 12, 40.0, 0),       # ragged 16-token tiles, T > 2M-1
    ("f32", 1, 1, 50, 64, 4, 7, 7.0, 0),         # T = S = 2M-1 (sliding window)
    ("f32", 2, 1, 33, 32, 4, 5, 20.0, 9),        # later start position
    ("bf16", 1, 2, 300, 128, 64, 64, 1024.0, 0), # the LM-layer (M, S, T), shortened
    # the chunked backward (32-token chunks, d in {64, 128}, S in {32, 64}):
    ("bf16", 1, 2, 150, 64, 17, 32, 33.0, 0),    # T = 2M-1: exact zeros of 1 - D
    ("bf16", 2, 1, 77, 128, 32, 64, 512.0, 45),  # ragged last chunk, later start position
    ("bf16", 1, 1, 1000, 64, 64, 64, 1024.0, 0), # 32 chunks
    ("bf16", 3, 1, 16, 128, 16, 32, 64.0, 0),    # half a chunk
])
def test_backward_against_oracle_vjp(orc, dtype, B, H, L, d, M, S, T, pos0):
    """dq, dk, dv of the decayed forward against the oracle's VJP of Alg. 1 with decay."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    dev = require_cuda()
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    q, k, v = make_qkv(B, H, L, d, dtype=dtype, seed=L + S)
    do = make_dout(B, H, L, d, dtype=dtype, seed=L + S)
    tq, tk, tv, tdo = (to_dev(x, dev, tdt) for x in (q, k, v, do))
    o, lse, _ = bla.bla_decay_forward(tq, tk, tv, M, S, T, pos0=pos0)
    got = bla.bla_decay_backward(tq, tk, tv, o, tdo, lse, M, S, T, pos0=pos0)
    bla.bla_device_error()
    ref = orc.backward_decay(q, k, v, do, M, S, T, pos0=pos0)
    tol = 1e-4 if dtype == "f32" else TOL_GRAD
    for name, a, b in zip(("dq", "dk", "dv"), got, ref):
        assert rel(a.float().cpu().numpy(), b) <= tol, (name, rel(a.float().cpu().numpy(), b))


def test_empty_sequence_passes_state_through():
    """L = 0: nothing to attend; the final state is the given one (or zero without one)."""
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    z = torch.zeros((1, 2, 0, 32), device=dev)
    st0 = torch.randn((1, 2, 2, 5, 32), device=dev)
    st = st0.clone()
    o, _, out = bla.bla_decay_forward(z, z, z, 3, 5, 9.0, pos0=4, state=st, want_state=True)
    _, _, zero = bla.bla_decay_forward(z, z, z, 3, 5, 9.0, want_state=True)
    bla.bla_device_error()
    assert o.shape == (1, 2, 0, 32)
    assert torch.equal(out, st0)
    assert float(zero.abs().max()) == 0.0


def test_chunked_backward_per_head_periods(orc):
    """The chunked backward with one period per head (one D_M table and grid per head)."""
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_dout, make_qkv
    dev = require_cuda()
    TH = [33.0, 256.0, 700.5]
    B, H, L, d, M, S = 2, 3, 130, 64, 17, 32
    q, k, v = make_qkv(B, H, L, d, dtype="bf16", seed=41)
    do = make_dout(B, H, L, d, dtype="bf16", seed=41)
    tq, tk, tv, tdo = (to_dev(x, dev, torch.bfloat16) for x in (q, k, v, do))
    o, lse, _ = bla.bla_decay_forward(tq, tk, tv, M, S, TH)
    got = bla.bla_decay_backward(tq, tk, tv, o, tdo, lse, M, S, TH)
    bla.bla_device_error()
    ref = orc.backward_decay(q, k, v, do, M, S, TH)
    for name, a, r in zip(("dq", "dk", "dv"), got, ref):
        a = a.float().cpu().numpy()
        assert rel(a, r) <= TOL_GRAD, (name, rel(a, r))
        # rows are compared within their head: heads at different periods have gradients of different sizes
        for b in range(B):
            for h in range(H):
                worst = row_errors(a[b, h], r[b, h])[1]
                assert worst <= TOL_GRAD, (name, b, h, worst)
