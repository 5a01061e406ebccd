"""Float64 CPU oracle for Blurry Window Attention (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg may import
this package.  The CUDA product path never imports, links or executes it.
"""
from .oracle import (  # noqa: F401
    FORMS, tables, dirichlet, forward, forward_decay, backward, backward_decay, period, omega_of, max_threads,
)
