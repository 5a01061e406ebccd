"""Seeded synthetic inputs for Blurry Window Attention workloads.

This module is shared by the tests, the bench and the oracle checks.  It holds
no arithmetic of the method itself: it only draws seeded random numbers with
the shapes and distributions of the workloads below and rounds them to the
storage dtype (bf16, round-to-nearest-even) so that the CUDA path and the
float64 oracle consume exactly the same values.

Every draw uses numpy's PCG64 generator seeded through SeedSequence(seed)
spawned into independent streams: q, k, v, upstream gradient, initial state
and duplicate-key positions.
"""
from dataclasses import dataclass, field

import numpy as np

STREAMS = ("q", "k", "v", "dout", "state", "dup", "x", "w")


@dataclass(frozen=True)
class Workload:
    """One synthetic BLA workload (sizes, mode count, slots, period)."""
    name: str
    dtype: str          # "f32" or "bf16": storage dtype of q, k, v, o
    B: int
    H: int
    L: int
    d: int
    M: int
    S: int
    T: float            # period ("window")
    chunk: int          # chunk length used for FLOP accounting
    recall_dup: float = 0.0   # fraction of keys copied from a random earlier position
    backward: bool = False
    decode_steps: int = 0     # >0: single-token decode workload
    decode_pos0: int = 0
    state_std: float = 0.0
    notes: str = field(default="", compare=False)


WORKLOADS = {
    "fwd_f32_small": Workload("fwd_f32_small", "f32", B=1, H=2, L=256, d=32, M=16, S=16, T=64, chunk=64,
                              notes="fp32 forward; q,k,v ~ N(0,1)/sqrt(d); seed 0"),
    "fwd_bf16_recall": Workload("fwd_bf16_recall", "bf16", B=64, H=4, L=512, d=64, M=32, S=32, T=256,
                                chunk=128, recall_dup=0.10,
                                notes="recall-shaped: 10% of keys duplicated at earlier positions"),
    "fwdbwd_bf16_lm": Workload("fwdbwd_bf16_lm", "bf16", B=8, H=8, L=4096, d=128, M=64, S=64, T=1024,
                               chunk=128, backward=True,
                               notes="LM-layer shape, model dim 1024; upstream grad ~ N(0,1)"),
    "prefill_bf16_long": Workload("prefill_bf16_long", "bf16", B=1, H=16, L=65536, d=128, M=128, S=128,
                                  T=4096, chunk=128, notes="long-context prefill"),
    # a BLA layer of the RegBench-sized LM (model dim 128, 4 heads, batch 32; M = 16 of the searched
    # 8..64, S = 2M-1 slots, T = 2(2M-1) of the searched [1, 2, 4](2M-1)); the sequence length is
    # not stated, 256 is assumed.  Odd S and d = 32 run on the fp32 path.
    "lm_block_f32": Workload("lm_block_f32", "f32", B=32, H=4, L=256, d=32, M=16, S=31, T=62, chunk=64,
                             notes="x ~ N(0,1) [B, L, 128]; W_q, W_k, W_v, W_o ~ N(0, 1/128)"),
    "decode_bf16": Workload("decode_bf16", "bf16", B=256, H=16, L=1, d=128, M=128, S=128, T=4096,
                            chunk=1, decode_steps=1024, decode_pos0=4096, state_std=0.1,
                            notes="single-token decode, fp32 state ~ N(0, 0.1^2)"),
    # the state decay of Sec. 3.3 (absolute form): the LM-layer prefill shape, and the decode shape
    # with a random slot-space state [B, H, 2, S, d]
    "decay_bf16_lm": Workload("decay_bf16_lm", "bf16", B=8, H=8, L=4096, d=128, M=64, S=64, T=1024,
                              chunk=128, notes="LM-layer shape with state decay; q,k,v ~ N(0,1)/sqrt(d)"),
    "decay_decode_bf16": Workload("decay_decode_bf16", "bf16", B=256, H=16, L=1, d=128, M=128, S=128,
                                  T=4096, chunk=1, decode_steps=1, decode_pos0=4096, state_std=0.1,
                                  notes="decode with state decay, fp32 slot state ~ N(0, 0.1^2)"),
}


def bf16_round(x) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = a.view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    out = (r << 16).astype(np.uint32).view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out = out.copy()
        out[nan] = np.nan
    return out


def bf16_bits(x) -> np.ndarray:
    """The uint16 bit patterns of bf16-representable float32 values."""
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    return (a.view(np.uint32) >> 16).astype(np.uint16)


def _streams(seed: int):
    seqs = np.random.SeedSequence(seed).spawn(len(STREAMS))
    return {n: np.random.Generator(np.random.PCG64(s)) for n, s in zip(STREAMS, seqs)}


def _store(x, dtype):
    x = np.asarray(x, dtype=np.float32)
    return bf16_round(x) if dtype == "bf16" else x


def make_qkv(B, H, L, d, dtype="bf16", seed=0, sharp=False, recall_dup=0.0, dv=None):
    """q, k, v as float32 arrays [B, H, L, d] holding values exactly representable in ``dtype``.

    Default scaling is N(0,1)/sqrt(d).  ``sharp`` draws q and k as N(0,1)
    (no 1/sqrt(d)), which makes the slot softmax peaked.  ``recall_dup`` copies
    that fraction of key positions t (distinct, in [1, L)) from a uniformly drawn
    earlier position t' < t, forming key-value pairs; values stay independent.
    """
    dv = d if dv is None else dv
    g = _streams(seed)
    qk_div = 1.0 if sharp else np.sqrt(d)
    q = g["q"].standard_normal((B, H, L, d)) / qk_div
    k = g["k"].standard_normal((B, H, L, d)) / qk_div
    v = g["v"].standard_normal((B, H, L, dv)) / np.sqrt(dv)
    if recall_dup > 0.0 and L > 1:
        n = int(np.floor(recall_dup * L))
        for b in range(B):
            for h in range(H):
                pos = np.sort(g["dup"].choice(np.arange(1, L), size=n, replace=False))
                for t in pos:
                    src = int(g["dup"].integers(0, t))
                    k[b, h, t] = k[b, h, src]
    return _store(q, dtype), _store(k, dtype), _store(v, dtype)


def make_dout(B, H, L, dv, dtype="bf16", seed=0):
    """Upstream gradient dO ~ N(0, 1), [B, H, L, dv]."""
    g = _streams(seed)
    return _store(g["dout"].standard_normal((B, H, L, dv)), dtype)


def make_state(B, H, M, d, std=0.1, seed=0):
    """Random fp32 recurrent state [B, H, 2, M, 2, d] ~ N(0, std^2); sin row of mode 0 is zero."""
    g = _streams(seed)
    st = (g["state"].standard_normal((B, H, 2, M, 2, d)) * std).astype(np.float32)
    st[:, :, :, 0, 1, :] = 0.0
    return st


def make_slot_state(B, H, S, d, std=0.1, seed=0):
    """Random fp32 slot-space state [B, H, 2, S, d] ~ N(0, std^2) (the decayed form's state)."""
    g = _streams(seed)
    return (g["state"].standard_normal((B, H, 2, S, d)) * std).astype(np.float32)


def make_decode_step(step, B, H, d, dtype="bf16", seed=0):
    """q, k, v of one decode step, [B, H, d] each, N(0,1)/sqrt(d).

    Each step draws from its own stream, SeedSequence([seed, step]), so any step
    can be regenerated alone without materialising the whole run.
    """
    seqs = np.random.SeedSequence([int(seed), int(step)]).spawn(3)
    g = [np.random.Generator(np.random.PCG64(s)) for s in seqs]
    q = g[0].standard_normal((B, H, d)) / np.sqrt(d)
    k = g[1].standard_normal((B, H, d)) / np.sqrt(d)
    v = g[2].standard_normal((B, H, d)) / np.sqrt(d)
    return _store(q, dtype), _store(k, dtype), _store(v, dtype)


def workload_inputs(w: Workload, seed=0, sharp=False):
    """The seeded inputs of a workload as a dict of float32 numpy arrays."""
    if w.decode_steps:
        q, k, v = make_decode_step(0, w.B, w.H, w.d, w.dtype, seed)
        return {"q": q, "k": k, "v": v, "state": make_state(w.B, w.H, w.M, w.d, w.state_std, seed)}
    q, k, v = make_qkv(w.B, w.H, w.L, w.d, w.dtype, seed, sharp=sharp, recall_dup=w.recall_dup)
    out = {"q": q, "k": k, "v": v}
    if w.backward:
        out["dout"] = make_dout(w.B, w.H, w.L, w.d, w.dtype, seed)
    return out


def make_block_inputs(B, L, dm, seed=0):
    """Input activations x ~ N(0, 1) [B, L, dm] and projection weights W_q, W_k, W_v, W_o ~
    N(0, 1/dm) [dm, dm] for one LM-block layer (float32)."""
    st = _streams(seed)
    sx, sw = st["x"], st["w"]
    x = sx.standard_normal((B, L, dm)).astype(np.float32)
    ws = [(sw.standard_normal((dm, dm)) / np.sqrt(dm)).astype(np.float32) for _ in range(4)]
    return x, ws
