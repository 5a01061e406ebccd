"""Thin ctypes binding of libbla_gb300.so (C ABI in include/bla.h).

The functions keep the C names.  They only marshal arguments: take torch CUDA
tensors (PyTorch supplies device memory and streams), allocate outputs and the
workspace with torch, pass raw pointers and the current stream to the library,
and raise BlaError on any non-OK status.  All computation happens in the CUDA
library; if it is missing this module raises instead of falling back.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbla_gb300.so")

BLA_OK, BLA_ERR_INVALID, BLA_ERR_UNSUPPORTED, BLA_ERR_CUDA, BLA_ERR_TIMEOUT = range(5)
BLA_F32, BLA_BF16 = 0, 1
BLA_WS_FORWARD, BLA_WS_BACKWARD, BLA_WS_DECODE, BLA_WS_FORWARD_HOST = 0, 1, 2, 3
BLA_WS_DECAY_FORWARD, BLA_WS_DECAY_DECODE, BLA_WS_DECAY_BACKWARD = 4, 5, 6
BLA_PHASE_LAG, BLA_PHASE_ABSOLUTE = 0, 1
PHASE_MODES = {"lag": BLA_PHASE_LAG, "absolute": BLA_PHASE_ABSOLUTE}

EXPORTED = ("bla_workspace_bytes", "bla_forward_chunked", "bla_decode_step", "bla_backward",
            "bla_device_error", "bla_status_string", "bla_last_error_string", "bla_kernel_launches",
            "bla_profile_enable", "bla_profile_collect", "bla_decode_step_noalloc", "bla_forward_chunked_host",
            "bla_selftest_wait_timeout", "bla_decay_forward", "bla_decay_decode_step",
            "bla_decay_backward")

# bla_kernel_id
KERNELS = ("tables", "tables_bf16", "prepass", "scan", "kpass", "vpass", "fwd_f32", "decode", "bwd", "decay")


class BlaError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s (status %d)" % (msg, status))
        self.status = status


class Params(ctypes.Structure):
    """Mirror of bla_params."""
    _fields_ = [("B", ctypes.c_int), ("H", ctypes.c_int), ("L", ctypes.c_int),
                ("d_k", ctypes.c_int), ("d_v", ctypes.c_int), ("M", ctypes.c_int), ("S", ctypes.c_int),
                ("window", ctypes.c_double), ("omega", ctypes.c_double), ("chunk", ctypes.c_int),
                ("scale", ctypes.c_double), ("dtype", ctypes.c_int), ("phase_mode", ctypes.c_int),
                ("periods", ctypes.POINTER(ctypes.c_double))]


_lib = None


def load():
    """Load the CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("libbla_gb300.so is missing at %s; run __graft_entry__.build() "
                           "(there is no CPU fallback)" % LIB_PATH)
    lib = ctypes.CDLL(LIB_PATH)
    vp, sz, P = ctypes.c_void_p, ctypes.c_size_t, ctypes.POINTER(Params)
    lib.bla_workspace_bytes.restype = sz
    lib.bla_workspace_bytes.argtypes = [P, ctypes.c_int]
    lib.bla_forward_chunked.restype = ctypes.c_int
    lib.bla_forward_chunked.argtypes = [P, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_selftest_wait_timeout.restype = ctypes.c_int
    lib.bla_selftest_wait_timeout.argtypes = [ctypes.c_int, vp]
    lib.bla_forward_chunked_host.restype = ctypes.c_int
    lib.bla_forward_chunked_host.argtypes = [P, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_decode_step.restype = ctypes.c_int
    lib.bla_decode_step.argtypes = [P, ctypes.c_longlong, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_decode_step_noalloc.restype = ctypes.c_int
    lib.bla_decode_step_noalloc.argtypes = [P, ctypes.c_longlong, vp, vp, vp, vp, vp, vp]
    lib.bla_decay_forward.restype = ctypes.c_int
    lib.bla_decay_forward.argtypes = [P, ctypes.c_longlong, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_decay_decode_step.restype = ctypes.c_int
    lib.bla_decay_decode_step.argtypes = [P, ctypes.c_longlong, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_decay_backward.restype = ctypes.c_int
    lib.bla_decay_backward.argtypes = [P, ctypes.c_longlong, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_backward.restype = ctypes.c_int
    lib.bla_backward.argtypes = [P, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bla_device_error.restype = ctypes.c_int
    lib.bla_device_error.argtypes = [vp]
    lib.bla_status_string.restype = ctypes.c_char_p
    lib.bla_status_string.argtypes = [ctypes.c_int]
    lib.bla_last_error_string.restype = ctypes.c_char_p
    lib.bla_last_error_string.argtypes = []
    lib.bla_kernel_launches.restype = ctypes.c_longlong
    lib.bla_kernel_launches.argtypes = []
    lib.bla_profile_enable.restype = ctypes.c_int
    lib.bla_profile_enable.argtypes = [ctypes.c_int]
    lib.bla_profile_collect.restype = ctypes.c_int
    lib.bla_profile_collect.argtypes = [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)]
    _lib = lib
    return lib


def _check(status):
    if status != BLA_OK:
        lib = load()
        msg = lib.bla_last_error_string().decode() or lib.bla_status_string(status).decode()
        raise BlaError(status, msg)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(dt):
    if dt == torch.float32:
        return BLA_F32
    if dt == torch.bfloat16:
        return BLA_BF16
    raise BlaError(BLA_ERR_INVALID, "dtype must be float32 or bfloat16, got %s" % dt)


def _phase_code(phase_mode):
    if isinstance(phase_mode, str):
        if phase_mode not in PHASE_MODES:
            raise BlaError(BLA_ERR_INVALID, "phase_mode must be one of %s, got %r" % (sorted(PHASE_MODES), phase_mode))
        return PHASE_MODES[phase_mode]
    return int(phase_mode)


def make_params(B, H, L, d_k, d_v, M, S, window, omega=0.0, chunk=0, scale=0.0, dtype=torch.bfloat16,
                phase_mode="lag"):
    """bla_params; phase_mode is "lag" (Alg. 2, the default) or "absolute" (Alg. 1), or its code.

    ``window`` is the period T, or a sequence of H periods, one per head (Alg. 1 and Alg. 3 take
    T in R^H), passed as ``periods``."""
    periods = None
    if isinstance(window, (list, tuple)) or (hasattr(window, "__len__") and not isinstance(window, str)):
        vals = [float(x) for x in window]
        if len(vals) != int(H):
            raise BlaError(BLA_ERR_INVALID, "per-head periods need %d values, got %d" % (int(H), len(vals)))
        periods = (ctypes.c_double * len(vals))(*vals)
        window = max(vals)
    p = Params(int(B), int(H), int(L), int(d_k), int(d_v), int(M), int(S), float(window), float(omega),
               int(chunk), float(scale), _dtype_code(dtype), _phase_code(phase_mode))
    if periods is not None:
        p.periods = periods       # ctypes keeps the array alive with the structure
    return p


def bla_workspace_bytes(params, which):
    return int(load().bla_workspace_bytes(ctypes.byref(params), int(which)))


def _workspace(params, which, device, workspace):
    n = bla_workspace_bytes(params, which)
    if workspace is not None:
        return workspace, workspace.numel() * workspace.element_size()
    if n == 0:
        return None, 0
    return torch.empty(n, dtype=torch.uint8, device=device), n


def _need_cuda(*ts):
    for t in ts:
        if t is not None and (not t.is_cuda or not t.is_contiguous()):
            raise BlaError(BLA_ERR_INVALID, "tensors must be contiguous CUDA tensors")


def bla_forward_chunked(q, k, v, M, S, window, omega=0.0, chunk=0, scale=0.0, want_lse=True,
                        want_state=False, workspace=None, out=None, stream=None, phase_mode="lag"):
    """Chunked forward over q, k: [B,H,L,d_k], v: [B,H,L,d_v] (float32 or bfloat16 CUDA tensors).

    Returns (o, lse or None, state or None); state is [B,H,2,M,2,d] fp32 (needs d_k == d_v).
    """
    _need_cuda(q, k, v)
    B, H, L, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, L, dk, dv, M, S, window, omega, chunk, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, L, dv), dtype=q.dtype, device=q.device)
    lse = torch.empty((B, H, L), dtype=torch.float32, device=q.device) if want_lse else None
    st = torch.empty((B, H, 2, M, 2, dk), dtype=torch.float32, device=q.device) if want_state else None
    ws, n = _workspace(p, BLA_WS_FORWARD, q.device, workspace)
    _check(load().bla_forward_chunked(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(st),
                                      _ptr(ws), n, _stream(stream)))
    return o, lse, st


def bla_decode_step(q, k, v, state, pos, M, S, window, omega=0.0, scale=0.0, workspace=None, out=None,
                    stream=None, phase_mode="lag"):
    """One decode step; q, k, v: [B,H,d]; state [B,H,2,M,2,d] fp32 is updated in place. Returns o."""
    _need_cuda(q, k, v, state)
    B, H, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, 1, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    ws, n = _workspace(p, BLA_WS_DECODE, q.device, workspace)
    _check(load().bla_decode_step(ctypes.byref(p), int(pos), _ptr(q), _ptr(k), _ptr(v), _ptr(state), _ptr(o),
                                  _ptr(ws), n, _stream(stream)))
    return o


def bla_decode_step_noalloc(q, k, v, state, pos, M, S, window, omega=0.0, scale=0.0, out=None, stream=None,
                            phase_mode="lag"):
    """bla_decode_step without a workspace: the library's own fixed device scratch holds the
    tables, so the call allocates nothing (the output is allocated here unless `out` is given)."""
    _need_cuda(q, k, v, state)
    B, H, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, 1, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    _check(load().bla_decode_step_noalloc(ctypes.byref(p), int(pos), _ptr(q), _ptr(k), _ptr(v), _ptr(state),
                                          _ptr(o), _stream(stream)))
    return o


def bla_backward(q, k, v, o, dout, lse, M, S, window, omega=0.0, scale=0.0, workspace=None, stream=None,
                 phase_mode="lag"):
    """Gradients (dq, dk, dv) of the chunked forward for upstream gradient dout."""
    _need_cuda(q, k, v, o, dout, lse)
    B, H, L, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, L, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    dq, dkk, dvv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    ws, n = _workspace(p, BLA_WS_BACKWARD, q.device, workspace)
    _check(load().bla_backward(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(dout), _ptr(lse),
                               _ptr(dq), _ptr(dkk), _ptr(dvv), _ptr(ws), n, _stream(stream)))
    return dq, dkk, dvv


def bla_decay_forward(q, k, v, M, S, window, omega=0.0, scale=0.0, pos0=0, state=None, want_lse=True,
                      want_state=False, workspace=None, out=None, stream=None, phase_mode="absolute"):
    """Forward of Alg. 1 with the state decay of Sec. 3.3 over q, k: [B,H,L,d], v: [B,H,L,d].

    ``state`` (optional, [B,H,2,S,d] fp32) is the slot-space state the tokens continue from at
    absolute index ``pos0``.  Returns (o, lse or None, final state or None); with want_state and
    a given ``state``, the state is updated in place and returned."""
    _need_cuda(q, k, v, state)
    B, H, L, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, L, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, L, dv), dtype=q.dtype, device=q.device)
    lse = torch.empty((B, H, L), dtype=torch.float32, device=q.device) if want_lse else None
    st_out = None
    if want_state:
        st_out = state if state is not None else torch.empty((B, H, 2, S, dk), dtype=torch.float32, device=q.device)
    ws, n = _workspace(p, BLA_WS_DECAY_FORWARD, q.device, workspace)
    _check(load().bla_decay_forward(ctypes.byref(p), int(pos0), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse),
                                    _ptr(state), _ptr(st_out), _ptr(ws), n, _stream(stream)))
    return o, lse, st_out


def bla_decay_decode_step(q, k, v, state, pos, M, S, window, omega=0.0, scale=0.0, workspace=None, out=None,
                          stream=None, phase_mode="absolute"):
    """One decode step of the decayed form; q, k, v: [B,H,d]; state [B,H,2,S,d] fp32 is updated in
    place.  Returns o."""
    _need_cuda(q, k, v, state)
    B, H, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, 1, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, dv), dtype=q.dtype, device=q.device)
    ws, n = _workspace(p, BLA_WS_DECAY_DECODE, q.device, workspace)
    _check(load().bla_decay_decode_step(ctypes.byref(p), int(pos), _ptr(q), _ptr(k), _ptr(v), _ptr(state), _ptr(o),
                                        _ptr(ws), n, _stream(stream)))
    return o


def bla_decay_backward(q, k, v, o, dout, lse, M, S, window, omega=0.0, scale=0.0, pos0=0, workspace=None,
                       stream=None, phase_mode="absolute"):
    """Gradients (dq, dk, dv) of bla_decay_forward (zero initial state, tokens from pos0) for
    upstream gradient dout; o and lse are the forward's outputs."""
    _need_cuda(q, k, v, o, dout, lse)
    B, H, L, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, L, dk, dv, M, S, window, omega, 0, scale, q.dtype, phase_mode)
    dq, dkk, dvv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    ws, n = _workspace(p, BLA_WS_DECAY_BACKWARD, q.device, workspace)
    _check(load().bla_decay_backward(ctypes.byref(p), int(pos0), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(dout),
                                     _ptr(lse), _ptr(dq), _ptr(dkk), _ptr(dvv), _ptr(ws), n, _stream(stream)))
    return dq, dkk, dvv


def bla_device_error(stream=None):
    """Synchronise and raise BlaError if a bounded device wait gave up."""
    _check(load().bla_device_error(_stream(stream)))


def bla_selftest_wait_timeout(limit_ms=20, stream=None):
    """Launch the library's failure-path self-test (a bounded wait that runs out); the next
    bla_device_error() raises BlaError with status BLA_ERR_TIMEOUT."""
    _check(load().bla_selftest_wait_timeout(int(limit_ms), _stream(stream)))


def bla_kernel_launches():
    """Kernels this library has launched in this process."""
    return int(load().bla_kernel_launches())


def bla_profile_enable(on=True):
    """Record a CUDA event pair around every launch (on the launch stream) from now on."""
    _check(load().bla_profile_enable(1 if on else 0))


def bla_profile_collect():
    """{kernel name: (total ms, launches)} for the launches recorded since the last collect."""
    n = len(KERNELS)
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int * n)()
    _check(load().bla_profile_collect(ms, cnt))
    return {KERNELS[i]: (float(ms[i]), int(cnt[i])) for i in range(n) if cnt[i] > 0}


def _need_host(*ts):
    for t in ts:
        if t.is_cuda or not t.is_contiguous():
            raise BlaError(BLA_ERR_INVALID, "host tensors must be contiguous CPU tensors")


def bla_forward_chunked_host(q, k, v, M, S, window, omega=0.0, chunk=0, scale=0.0, out=None, workspace=None,
                             stream=None, phase_mode="lag", device=None):
    """bla_forward_chunked_host: q, k, v and the returned o are CPU tensors (page-locked for the
    copies to overlap the compute).  `workspace` is a CUDA uint8 tensor of at least
    bla_workspace_bytes(params, BLA_WS_FORWARD_HOST) bytes (allocated if None).  o is complete once
    `stream` (default: the current stream) has been synchronised."""
    _need_host(q, k, v)
    B, H, L, dk = q.shape
    dv = v.shape[-1]
    p = make_params(B, H, L, dk, dv, M, S, window, omega, chunk, scale, q.dtype, phase_mode)
    o = out if out is not None else torch.empty((B, H, L, dv), dtype=q.dtype, pin_memory=True)
    _need_host(o)
    dev = torch.device("cuda") if device is None else device
    ws, n = _workspace(p, BLA_WS_FORWARD_HOST, dev, workspace)
    _check(load().bla_forward_chunked_host(ctypes.byref(p), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(ws), n,
                                           _stream(stream)))
    return o


def forward_from_host(q_host, k_host, v_host, M, S, window, omega=0.0, scale=0.0, device=None, bufs=None,
                      out_host=None, stream=None, phase_mode="lag"):
    """bla_forward_chunked_host with the workspace (and the output, if `out_host` is None) cached in
    the dict `bufs` between calls.  Returns the host output; it is complete once the stream has
    been synchronised."""
    dev = torch.device("cuda") if device is None else device
    bufs = {} if bufs is None else bufs
    B, H, L, dk = q_host.shape
    dv = v_host.shape[-1]
    # every argument the workspace size may depend on (per-head periods as a tuple)
    per = tuple(float(x) for x in window) if hasattr(window, "__len__") else float(window)
    key = (B, H, L, dk, dv, M, S, per, float(omega), float(scale), q_host.dtype, phase_mode)
    if bufs.get("key") != key:
        p = make_params(B, H, L, dk, dv, M, S, window, omega, 0, scale, q_host.dtype, phase_mode)
        bufs["ws"] = torch.empty(max(bla_workspace_bytes(p, BLA_WS_FORWARD_HOST), 1), dtype=torch.uint8, device=dev)
        bufs["key"] = key
    if out_host is None:
        if "o" not in bufs or bufs["o"].shape != (B, H, L, dv) or bufs["o"].dtype != q_host.dtype:
            bufs["o"] = torch.empty((B, H, L, dv), dtype=q_host.dtype, pin_memory=True)
        out_host = bufs["o"]
    return bla_forward_chunked_host(q_host, k_host, v_host, M, S, window, omega, 0, scale, out=out_host,
                                    workspace=bufs["ws"], stream=stream, phase_mode=phase_mode, device=dev)
