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
