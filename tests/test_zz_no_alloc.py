"""bla_decode_step_noalloc: the decode step for callers that may not allocate device memory.

Such callers (a serving plugin with a fixed memory budget, a token loop that must not call
the allocator mid-step) pass no workspace; the tables live in the library's own fixed
device array.  The entry point is called through the C ABI with preallocated buffers and
must reproduce the regular bla_decode_step (which uses a caller workspace) on two
consecutive steps.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest

from gpu_util import TOL_BF16, rel, require_cuda, to_dev


@pytest.mark.gpu
def test_noalloc_decode_matches_workspace_decode_twice():
    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import make_decode_step, make_state
    dev = require_cuda()
    lib = bla.load()
    B, H, d, M, S, T, pos0 = 8, 4, 128, 64, 64, 512.0, 600
    st0 = torch.from_numpy(make_state(B, H, M, d, std=0.1, seed=5)).to(dev)
    st_ref, st_new = st0.clone(), st0.clone()
    p = bla.make_params(B, H, 1, d, d, M, S, T, dtype=torch.bfloat16)
    ws = torch.empty(bla.bla_workspace_bytes(p, bla.BLA_WS_DECODE), dtype=torch.uint8, device=dev)
    o_ref = torch.empty((B, H, d), dtype=torch.bfloat16, device=dev)
    o_new = torch.empty_like(o_ref)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for step in range(2):
        q, k, v = (to_dev(x, dev, torch.bfloat16) for x in make_decode_step(step, B, H, d, "bf16", seed=5))
        args = (ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()), ctypes.c_void_p(v.data_ptr()))
        r = lib.bla_decode_step(ctypes.byref(p), pos0 + step, *args, ctypes.c_void_p(st_ref.data_ptr()),
                                ctypes.c_void_p(o_ref.data_ptr()), ctypes.c_void_p(ws.data_ptr()), ws.numel(), stream)
        assert r == bla.BLA_OK
        r = lib.bla_decode_step_noalloc(ctypes.byref(p), pos0 + step, *args, ctypes.c_void_p(st_new.data_ptr()),
                                        ctypes.c_void_p(o_new.data_ptr()), stream)
        assert r == bla.BLA_OK, lib.bla_last_error_string()
        torch.cuda.synchronize()
        assert rel(o_new.float().cpu().numpy(), o_ref.float().cpu().numpy()) <= TOL_BF16
        assert rel(st_new.cpu().numpy(), st_ref.cpu().numpy()) <= 1e-6
    bla.bla_device_error()


@pytest.mark.gpu
def test_noalloc_rejects_tables_beyond_the_static_scratch():
    import torch
    from paper_2606_09862_gb300 import bla
    dev = require_cuda()
    lib = bla.load()
    # S = 256 slots x 2M = 1024 state rows: 1 MiB of tables, more than the 512 KiB array
    p = bla.make_params(1, 1, 1, 64, 64, 512, 256, 4096.0, dtype=torch.bfloat16)
    buf = torch.zeros(1 << 20, dtype=torch.float32, device=dev)
    ptr = ctypes.c_void_p(buf.data_ptr())
    r = lib.bla_decode_step_noalloc(ctypes.byref(p), 0, ptr, ptr, ptr, ptr, ptr, None)
    assert r == bla.BLA_ERR_UNSUPPORTED
    assert b"static scratch" in lib.bla_last_error_string()
