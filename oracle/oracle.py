"""ctypes front end of the float64 BLA oracle (test infrastructure only).

All arithmetic lives in ``bla_oracle.c``; this module only marshals numpy
arrays.  Arrays are float64 with shape [B, H, L, d]; the recurrent state is
[B, H, 2 (K, V), M, 2 (cos, sin), d] (the sin row of mode 0 is always zero).

Forms (see the C header for the paper passage each follows):
  "naive"     Alg. 2 (naive recurrent BLA), slots materialised per token
  "modes"     same recurrence, read-out through the modes (Eq. conv exchange of sums)
  "parallel"  closed form of Eq. (states) with translated Dirichlet kernels
  "absolute"  Alg. 1 (efficient recurrent BLA, time-rolling slots); pins only
  forward_decay, backward_decay: Alg. 1 with the state decay of Sec. 3.3 (slot-space state) and its VJP
"""
import ctypes

import numpy as np

from . import build as _build

FORMS = {"naive": 0, "modes": 1, "parallel": 2, "absolute": 3}

_lib = None
_dp = ctypes.POINTER(ctypes.c_double)


def _configure(lib):
    lib.orc_period.restype = ctypes.c_double
    lib.orc_period.argtypes = [ctypes.c_int, ctypes.c_double]
    lib.orc_omega.restype = ctypes.c_double
    lib.orc_omega.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_double]
    lib.orc_dirichlet.restype = ctypes.c_double
    lib.orc_dirichlet.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_double]
    lib.orc_tables.restype = None
    lib.orc_tables.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_double,
                               _dp, _dp, _dp]
    lib.orc_forward.restype = ctypes.c_int
    lib.orc_forward.argtypes = [ctypes.c_int] * 7 + [ctypes.c_double] * 3 + [ctypes.c_longlong] + \
        [_dp] * 6 + [ctypes.c_void_p]
    lib.orc_backward.restype = ctypes.c_int
    lib.orc_backward.argtypes = [ctypes.c_int] * 7 + [ctypes.c_double] * 3 + [_dp] * 7
    lib.orc_forward_decay.restype = ctypes.c_int
    lib.orc_forward_decay.argtypes = [ctypes.c_int] * 6 + [ctypes.c_double] * 3 + [ctypes.c_longlong] + [_dp] * 6
    lib.orc_backward_decay.restype = ctypes.c_int
    lib.orc_backward_decay.argtypes = [ctypes.c_int] * 6 + [ctypes.c_double] * 3 + [ctypes.c_longlong] + [_dp] * 7
    lib.orc_max_threads.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    if _lib is None:
        _lib = _configure(ctypes.CDLL(_build.build()))
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_dp)


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def max_threads() -> int:
    """OpenMP threads the oracle's parallel loops use."""
    return int(_load().orc_max_threads())


def period(M: int, T: float) -> float:
    """Clamped period max(T, 2M-1) (Alg. 1 and Alg. 3)."""
    return float(_load().orc_period(int(M), float(T)))


def omega_of(M: int, T: float, omega: float = 0.0) -> float:
    """2*pi/T with the clamped period, unless omega > 0 is given (Sec. 3.1)."""
    return float(_load().orc_omega(int(M), float(T), float(omega)))


def dirichlet(M: int, x, omega: float) -> np.ndarray:
    """D_M(x) of Eq. (dirichlet) at angular frequency omega, elementwise."""
    lib = _load()
    xs = np.asarray(x, dtype=np.float64)
    return np.vectorize(lambda y: lib.orc_dirichlet(int(M), float(omega), float(y)))(xs)


def tables(M: int, S: int, T: float, omega: float = 0.0):
    """(delta, A, B): dilated time grid and Eq. (translated) coefficients, A/B of shape [S, M]."""
    delta = np.zeros(S)
    A = np.zeros((S, M))
    B = np.zeros((S, M))
    _load().orc_tables(int(M), int(S), float(T), float(omega), _ptr(delta), _ptr(A), _ptr(B))
    return delta, A, B


def _per_head(T, H):
    """The periods of Alg. 1 and Alg. 3 (T in R^H): None for one scalar period shared by every head,
    else the array of H periods (each head's grid, omega, A and B follow its own period)."""
    Ts = np.atleast_1d(np.asarray(T, dtype=np.float64))
    if Ts.size == 1 and np.ndim(T) == 0:
        return None
    if Ts.shape != (H,):
        raise ValueError("per-head periods need one value per head (%d), got shape %s" % (H, Ts.shape))
    return Ts


def _by_head(fn, Ts, arrays, H, **kw):
    """Run ``fn`` on each head's slice [:, h:h+1] at period Ts[h]; returns the per-head results."""
    out = []
    for h in range(H):
        sl = [None if a is None else np.asarray(a)[:, h:h + 1] for a in arrays]
        out.append(fn(*sl, T=float(Ts[h]), **kw))
    return out


def _cat_dicts(parts):
    res = {}
    for key in parts[0]:
        vals = [p[key] for p in parts]
        res[key] = None if vals[0] is None else np.concatenate(vals, axis=1)
    return res


def forward(q, k, v, M, S, T, omega=0.0, scale=0.0, form="naive", state=None, pos0=0,
            want=None, return_state=False):
    """Run the oracle forward.

    q, k: [B, H, L, dk]; v: [B, H, L, dv].  ``state`` (optional) is the initial
    recurrent state [B, H, 2, M, 2, d] (requires dk == dv for this packed
    layout) and ``pos0`` the absolute index of token 0 (slot mask t >= Delta_j).
    ``want`` (bool [L]) restricts which tokens get an output (others are NaN);
    the state always advances over every token.
    ``T`` is one period, or one per head (Alg. 1 and Alg. 3 take T in R^H).
    Returns dict(o=[B,H,L,dv], lse=[B,H,L], state=final state or None).
    """
    Ts = _per_head(T, np.shape(q)[1])
    if Ts is not None:
        parts = _by_head(lambda q_, k_, v_, st_, T: forward(q_, k_, v_, M, S, T, omega, scale, form, st_, pos0, want,
                                                             return_state),
                         Ts, (q, k, v, state), len(Ts))
        return _cat_dicts(parts)
    q, k, v = _f64(q), _f64(k), _f64(v)
    Bn, Hn, L, dk = q.shape
    dv = v.shape[-1]
    NH = Bn * Hn
    o = np.full((Bn, Hn, L, dv), np.nan)
    lse = np.full((Bn, Hn, L), np.nan)
    st = None
    if state is not None or return_state:
        if state is None:
            st = np.zeros((Bn, Hn, 2 * M * (dk + dv)))
        else:
            st = _f64(state).reshape(Bn, Hn, -1).copy()
            assert st.shape[-1] == 2 * M * (dk + dv)
    wm = None
    if want is not None:
        wm = np.ascontiguousarray(np.asarray(want, dtype=np.uint8))
        assert wm.shape == (L,)
    rc = _load().orc_forward(FORMS[form], NH, L, dk, dv, int(M), int(S), float(T), float(omega),
                             float(scale), int(pos0), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse),
                             _ptr(st), None if wm is None else wm.ctypes.data)
    if rc != 0:
        raise ValueError("oracle forward rejected its arguments (code %d)" % rc)
    out = {"o": o, "lse": lse, "state": None}
    if st is not None:
        if dk == dv:
            out["state"] = st.reshape(Bn, Hn, 2, M, 2, dk)
        else:
            out["state"] = st
    return out


def forward_decay(q, k, v, M, S, T, omega=0.0, scale=0.0, state=None, pos0=0, return_state=False):
    """Alg. 1 with the state decay of Sec. 3.3: K~[j] <- (1 - D_j(t)) K~[j] + D_j(t) k_t.

    q, k: [B, H, L, dk]; v: [B, H, L, dv].  ``state`` (optional) is the slot-space state
    [B, H, 2, S, d] (K~ then V~; any shape with S*(dk+dv) values per head) and ``pos0`` the
    absolute index of token 0.  Returns dict(o, lse, state) like ``forward``; the state is
    [B, H, 2, S, d] when dk == dv.  ``T`` is one period or one per head.
    """
    Ts = _per_head(T, np.shape(q)[1])
    if Ts is not None:
        parts = _by_head(lambda q_, k_, v_, st_, T: forward_decay(q_, k_, v_, M, S, T, omega, scale, st_, pos0,
                                                                   return_state),
                         Ts, (q, k, v, state), len(Ts))
        return _cat_dicts(parts)
    q, k, v = _f64(q), _f64(k), _f64(v)
    Bn, Hn, L, dk = q.shape
    dv = v.shape[-1]
    o = np.full((Bn, Hn, L, dv), np.nan)
    lse = np.full((Bn, Hn, L), np.nan)
    st = None
    if state is not None or return_state:
        st = np.zeros((Bn, Hn, S * (dk + dv))) if state is None else _f64(state).reshape(Bn, Hn, -1).copy()
        assert st.shape[-1] == S * (dk + dv)
    rc = _load().orc_forward_decay(Bn * Hn, L, dk, dv, int(M), int(S), float(T), float(omega), float(scale),
                                   int(pos0), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(st))
    if rc != 0:
        raise ValueError("oracle decay forward rejected its arguments (code %d)" % rc)
    out = {"o": o, "lse": lse, "state": None}
    if st is not None:
        out["state"] = st.reshape(Bn, Hn, 2, S, dk) if dk == dv else st
    return out


def backward(q, k, v, dout, M, S, T, omega=0.0, scale=0.0, form="parallel"):
    """Vector-Jacobian product (dq, dk, dv) of the forward for upstream gradient dout.

    ``form`` "parallel" (any of the lag-form forwards; they agree) or "absolute" (Alg. 1).
    ``T`` is one period or one per head."""
    Ts = _per_head(T, np.shape(q)[1])
    if Ts is not None:
        parts = _by_head(lambda q_, k_, v_, do_, T: backward(q_, k_, v_, do_, M, S, T, omega, scale, form),
                         Ts, (q, k, v, dout), len(Ts))
        return tuple(np.concatenate([p[i] for p in parts], axis=1) for i in range(3))
    if form not in ("parallel", "absolute"):
        raise ValueError("backward form must be 'parallel' or 'absolute', got %r" % (form,))
    q, k, v, dout = _f64(q), _f64(k), _f64(v), _f64(dout)
    Bn, Hn, L, dk = q.shape
    dv = v.shape[-1]
    dq = np.zeros_like(q)
    dkk = np.zeros_like(k)
    dvv = np.zeros_like(v)
    rc = _load().orc_backward(FORMS[form], Bn * Hn, L, dk, dv, int(M), int(S), float(T), float(omega), float(scale),
                              _ptr(q), _ptr(k), _ptr(v), _ptr(dout), _ptr(dq), _ptr(dkk), _ptr(dvv))
    if rc != 0:
        raise ValueError("oracle backward rejected its arguments (code %d)" % rc)
    return dq, dkk, dvv


def backward_decay(q, k, v, dout, M, S, T, omega=0.0, scale=0.0, pos0=0):
    """Vector-Jacobian product (dq, dk, dv) of ``forward_decay`` from the zero state, tokens at
    absolute indices pos0 .., for upstream gradient dout.  ``T`` is one period or one per head."""
    Ts = _per_head(T, np.shape(q)[1])
    if Ts is not None:
        parts = _by_head(lambda q_, k_, v_, do_, T: backward_decay(q_, k_, v_, do_, M, S, T, omega, scale, pos0),
                         Ts, (q, k, v, dout), len(Ts))
        return tuple(np.concatenate([p[i] for p in parts], axis=1) for i in range(3))
    q, k, v, dout = _f64(q), _f64(k), _f64(v), _f64(dout)
    Bn, Hn, L, dk = q.shape
    dv = v.shape[-1]
    dq, dkk, dvv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    rc = _load().orc_backward_decay(Bn * Hn, L, dk, dv, int(M), int(S), float(T), float(omega), float(scale),
                                    int(pos0), _ptr(q), _ptr(k), _ptr(v), _ptr(dout), _ptr(dq), _ptr(dkk), _ptr(dvv))
    if rc != 0:
        raise ValueError("oracle decay backward rejected its arguments (code %d)" % rc)
    return dq, dkk, dvv
