"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import numpy as np


def rel(a, b):
    """Relative L2 error ||a - b|| / ||b|| over the whole tensor (float64)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / nb) if nb > 0 else float(np.linalg.norm(a - b))


def require_cuda():
    import torch
    if not torch.cuda.is_available():
        raise RuntimeError("this test needs a CUDA GPU (run with -m 'not gpu' on CPU-only hosts)")
    return torch.device("cuda:0")


def to_dev(x, dev, dtype):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev).to(dtype)


TOL_F32 = 1e-4      # fp32 path (relative L2)
TOL_BF16 = 2e-2     # bf16 in / fp32 accumulate (relative L2)
TOL_GRAD = 3e-2     # gradients (relative L2)


def row_errors(a, b):
    """(pooled, worst_row): the relative L2 error of the whole tensor, and the largest per-row error
    ||a_row - b_row|| / max(||b_row||, median row norm) over every row of the last axis.

    The floor at the median row norm matters only for rows whose exact value vanishes (dq of the
    first token, whose softmax has one visible slot; dk of the last key): their absolute error is of
    the size of a typical row's, so it is measured against a typical row.  Pass one head at a time
    where heads differ in scale (per-head periods)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    d = a.shape[-1]
    a2, b2 = a.reshape(-1, d), b.reshape(-1, d)
    err = np.linalg.norm(a2 - b2, axis=1)
    nb = np.linalg.norm(b2, axis=1)
    floor = max(float(np.median(nb)), 1e-300)
    worst = float(np.max(err / np.maximum(nb, floor))) if err.size else 0.0
    return rel(a, b), worst


# Per-row bounds (bf16 paths).  Standard inputs, N(0,1)/sqrt(d): scores stay within a few units, so
# the bf16 roundings perturb each row about as much as the whole tensor and every row meets the
# tensor tolerance.  Sharp inputs (q, k ~ N(0,1)) reach |s| ~ 30: a score error ds moves a peaked
# softmax row by up to 2 |ds| max_j ||V~_j - o_t|| / ||o_t||, with |ds| up to the lse bound below
# (~7e-2) and a spread ratio near 0.7, so a row may move by up to ~1e-1.
TOL_ROW_BF16 = TOL_BF16
TOL_ROW_SHARP = 1e-1
# Gradient rows on sharp inputs: ds = p (dp - rowsum(dO o)) is linear in p, and a peaked row's p moves
# by up to 2 |ds| relative (the softmax Jacobian), ~0.15 at the score errors above; dq, dk and dv rows
# inherit that.
TOL_ROW_SHARP_GRAD = 0.15


def lse_bound(ref_lse):
    """Per-token bound on |lse - lse_ref| for bf16-in / fp32-accumulate paths.

    lse is 1-Lipschitz in the max-norm of the scores, so its error is at most the largest score
    error of a visible slot.  A score s_tj = scale * sum_r Y_tr PHI_jr is contracted from bf16
    operands: PHI and Y are rounded to bf16 (unit roundoff u = 2^-9 each), and Y is itself contracted
    from bf16 operands (2u more), so each product carries a relative error of at most 4u = 2^-7.
    Allowing a factor 4 for cancellation in the sum over modes (sum_r |Y PHI| against |s|) gives
    2^-5 of the score scale, which lse + 1 bounds from above for the slots that carry weight."""
    return 2.0 ** -5 * (np.abs(np.asarray(ref_lse, dtype=np.float64)) + 1.0)
