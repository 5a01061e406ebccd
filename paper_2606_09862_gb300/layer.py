"""A Blurry Window Attention layer inside an LM block (the token mixer of Sec. 3 between the
block's input and output projections).

q, k, v = x W_q, x W_k, x W_v, split into H heads of d = d_model / H; o = BLA(q, k, v) by the CUDA
library (bla_forward_chunked); y = concat_heads(o) W_o.  The four projections are plain GEMMs
(torch.matmul, i.e. cuBLAS); the mixing runs in the library's kernels.  fp32 activations use the
library's fp32 path (any M, S, d), bf16 activations its tensor-core path.
"""
from . import bla


def bla_block_forward(x, w_q, w_k, w_v, w_o, H, M, S, window, omega=0.0, phase_mode="lag", workspace=None):
    """x: [B, L, d_model] CUDA tensor; w_*: [d_model, d_model].  Returns y: [B, L, d_model]."""
    B, L, dm = x.shape
    if dm % H:
        raise bla.BlaError(bla.BLA_ERR_INVALID, "d_model (%d) must be a multiple of H (%d)" % (dm, H))
    d = dm // H

    def heads(t):
        return t.view(B, L, H, d).transpose(1, 2).contiguous()

    q, k, v = heads(x @ w_q), heads(x @ w_k), heads(x @ w_v)
    o, _, _ = bla.bla_forward_chunked(q, k, v, M, S, window, omega=omega, want_lse=False, workspace=workspace,
                                      phase_mode=phase_mode)
    return o.transpose(1, 2).reshape(B, L, dm) @ w_o
