"""Checks that pin the float64 oracle to facts fixed by the paper and by mathematics.

Each function returns the largest discrepancy it found (a float).  They are used
by test_oracle_pins.py against the real oracle and by test_oracle_mutants.py
against deliberately broken copies of it, to show that a plausible mistake in
the oracle (a sign, an index, a dropped term) makes at least one pin fail.

None of these functions calls the CUDA library.  The reference values are
computed here from closed forms that differ from the oracle's own formulas.
"""
import numpy as np


def rng(seed):
    return np.random.default_rng(seed)


def _worst(*vals):
    """Largest of the discrepancies; NaN counts as an infinite discrepancy."""
    out = 0.0
    for x in vals:
        x = float(x)
        if x != x:
            return float("inf")
        out = max(out, x)
    return out


def _softmax_masked(s, valid):
    s = np.where(valid, s, -np.inf)
    mx = s.max(axis=-1, keepdims=True)
    e = np.where(valid, np.exp(s - mx), 0.0)
    return e / e.sum(axis=-1, keepdims=True), (mx + np.log(e.sum(axis=-1, keepdims=True)))[..., 0]


def dirichlet_sine_ratio(M, w, x):
    """D_M(x) from the Dirichlet closed form: (2M-1) D_M(x) = sin((M-1/2) w x) / sin(w x / 2),
    i.e. sum_{m=-N}^{N} e^{i m y} = sin((N+1/2) y)/sin(y/2) at N = M-1, y = w x; value 1 where
    sin(w x / 2) = 0."""
    x = np.asarray(x, dtype=np.float64)
    den = np.sin(w * x / 2.0)
    num = np.sin((M - 0.5) * w * x)
    out = np.ones_like(x)
    nz = np.abs(den) > 1e-12
    out[nz] = num[nz] / ((2 * M - 1) * den[nz])
    return out


# ---------------------------------------------------------------- P1: kernel

def pin_dirichlet_identity(orc):
    """(2M-1) D_M(x) = sin((M-1/2)x)/sin(x/2) at omega = 1 (Eq. dirichlet; the identity
    sum_{m=-N}^{N} e^{imx} = sin((N+1/2)x)/sin(x/2) at N = M-1)."""
    err = 0.0
    xs = np.linspace(0.05, 2 * np.pi - 0.05, 97)
    for M in (1, 2, 3, 6, 17):
        d = orc.dirichlet(M, xs, 1.0)
        ref = np.sin((M - 0.5) * xs) / ((2 * M - 1) * np.sin(xs / 2))
        err = _worst(err, float(np.abs(d - ref).max()))
    return err


def pin_dirichlet_samples(orc):
    """D_M(0) = 1 and D_M(t) = 0 for t = 1..2M-2 at omega = 2 pi/(2M-1) (text after Eq. dirichlet)."""
    err = 0.0
    for M in (1, 2, 4, 9):
        n = 2 * M - 1
        d = orc.dirichlet(M, np.arange(n), 2 * np.pi / n)
        ref = np.zeros(n)
        ref[0] = 1.0
        err = _worst(err, float(np.abs(d - ref).max()))
    return err


# ------------------------------------------------------- grid and tables

def pin_grid(orc):
    """Dilated grid round(j T / S), half to even; the paper's grid at S = 2M-1; clamp T >= 2M-1."""
    err = 0.0
    delta, _, _ = orc.tables(3, 4, 10.0)
    err = _worst(err, float(np.abs(delta - np.array([0.0, 2.0, 5.0, 8.0])).max()))   # 2.5->2, 7.5->8
    M, T = 4, 14.0
    delta, _, _ = orc.tables(M, 2 * M - 1, T)
    ref = np.round(np.arange(2 * M - 1) / (2 * M - 1) * T)
    err = _worst(err, float(np.abs(delta - ref).max()))
    err = _worst(err, abs(orc.period(4, 3.0) - 7.0), abs(orc.period(4, 9.0) - 9.0))
    err = _worst(err, abs(orc.omega_of(4, 3.0) - 2 * np.pi / 7.0), abs(orc.omega_of(4, 3.0, 0.5) - 0.5))
    return err


def pin_translated_coefficients(orc):
    """App. B: D_M(t - Delta) = sum_m A[Delta,m] cos(m w t) + B[Delta,m] sin(m w t), with D_M
    from the sine-ratio closed form, for several periods (also T > 2M-1)."""
    err = 0.0
    for M, S, T in ((4, 7, 7.0), (4, 7, 14.0), (5, 6, 23.0), (3, 3, 11.0)):
        delta, A, B = orc.tables(M, S, T)
        w = 2 * np.pi / orc.period(M, T)
        t = np.arange(-30, 31, dtype=np.float64)
        m = np.arange(M)
        C = np.cos(np.outer(t, m) * w)
        Sn = np.sin(np.outer(t, m) * w)
        for j in range(S):
            lhs = dirichlet_sine_ratio(M, w, t - delta[j])
            rhs = C @ A[j] + Sn @ B[j]
            err = _worst(err, float(np.abs(lhs - rhs).max()))
    return err


# ------------------------------------------------------- P2: state closed form

def pin_state_closed_form(orc):
    """Eq. (states): after tokens 0..t, Kcos[m] = sum_{t'<=t} cos(m w (t-t')) k_t' and
    Ksin[m] = sum sin(m w (t-t')) k_t'; with an initial state Z0 the rotated Z0
    e^{i m w (t+1)} is added (App. B induction)."""
    g = rng(11)
    err = 0.0
    for M, S, T, L, d in ((3, 5, 5.0, 9, 4), (4, 3, 17.0, 13, 3)):
        q, k, v = (g.standard_normal((1, 2, L, d)) for _ in range(3))
        z0 = g.standard_normal((1, 2, 2, M, 2, d))
        z0[:, :, :, 0, 1, :] = 0.0
        w = 2 * np.pi / orc.period(M, T)
        for init in (None, z0):
            st = orc.forward(q, k, v, M, S, T, state=init, return_state=True)["state"]
            lag = (L - 1) - np.arange(L)
            for kv, x in ((0, k), (1, v)):
                for m in range(M):
                    zc = (np.cos(m * w * lag)[None, None, :, None] * x).sum(2)
                    zs = (np.sin(m * w * lag)[None, None, :, None] * x).sum(2)
                    if init is not None:
                        a, b = init[:, :, kv, m, 0], init[:, :, kv, m, 1]
                        ph = m * w * L
                        zc = zc + np.cos(ph) * a - np.sin(ph) * b
                        zs = zs + np.sin(ph) * a + np.cos(ph) * b
                    err = _worst(err, float(np.abs(st[:, :, kv, m, 0] - zc).max()),
                              float(np.abs(st[:, :, kv, m, 1] - zs).max()))
    return err


# ------------------------------------------------ P3: full resolution = attention

def pin_causal_attention(orc):
    """T = S = 2M-1 and L <= 2M-1 give causal softmax attention exactly (Fig. 2b; text after
    Eq. conv_key); lse is the log-sum-exp of the causal scores."""
    g = rng(5)
    err = 0.0
    for M, L, d in ((4, 7, 5), (6, 9, 3), (1, 1, 2)):
        n = 2 * M - 1
        q, k, v = (g.standard_normal((2, 1, L, d)) for _ in range(3))
        for form in ("naive", "modes", "parallel"):
            r = orc.forward(q, k, v, M, n, float(n), form=form)
            s = np.einsum("bhtd,bhud->bhtu", q, k) / np.sqrt(d)
            valid = np.tril(np.ones((L, L), bool))
            p, lse = _softmax_masked(s, valid)
            o = np.einsum("bhtu,bhud->bhtd", p, v)
            err = _worst(err, float(np.abs(r["o"] - o).max()), float(np.abs(r["lse"] - lse).max()))
    return err


# -------------------------------------------------- P4: aliasing modulo 2M-1

def pin_aliasing(orc):
    """T = S = 2M-1, L > 2M-1: slot j holds the sum of the keys k_t' with t - t' = j (mod 2M-1)
    (Eq. conv_key) and is visible once t >= j."""
    g = rng(7)
    err = 0.0
    for M, L, d in ((3, 17, 4), (4, 30, 2)):
        n = 2 * M - 1
        q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
        r = orc.forward(q, k, v, M, n, float(n), form="naive")
        for t in range(L):
            Ks = np.zeros((n, d))
            Vs = np.zeros((n, d))
            for u in range(t + 1):
                Ks[(t - u) % n] += k[0, 0, u]
                Vs[(t - u) % n] += v[0, 0, u]
            s = Ks @ q[0, 0, t] / np.sqrt(d)
            valid = np.arange(n) <= t
            p, _ = _softmax_masked(s[None], valid[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ Vs).max()))
    return err


# ------------------------------------------ blurry case (T > 2M-1, S != 2M-1)

def pin_blurry_bruteforce(orc):
    """T > 2M-1: slots are Dirichlet-blurred lags, K~_t[j] = sum_{t'<=t} D_M(t - t' - Delta_j) k_t'
    (Eq. compressed with Eq. translated), evaluated by brute force with the sine-ratio D_M and
    the grid round(j T/S) computed here."""
    g = rng(9)
    err = 0.0
    for M, S, T, L, d in ((3, 4, 10.0, 23, 3), (4, 6, 21.0, 40, 2), (2, 3, 8.0, 11, 5)):
        q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
        r = orc.forward(q, k, v, M, S, T, form="naive")
        w = 2 * np.pi / T
        delta = np.round(np.arange(S) * T / S)
        for t in range(L):
            u = np.arange(t + 1)
            W = dirichlet_sine_ratio(M, w, (t - u)[None, :] - delta[:, None])   # [S, t+1]
            Ks = W @ k[0, 0, : t + 1]
            Vs = W @ v[0, 0, : t + 1]
            s = Ks @ q[0, 0, t] / np.sqrt(d)
            valid = t >= delta
            p, lse = _softmax_masked(s[None], valid[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ Vs).max()),
                      float(abs(r["lse"][0, 0, t] - lse[0])))
    return err


# --------------------------------------------- P5: the oracle's forms agree

def pin_forms_agree(orc):
    """Alg. 2 recurrence = mode read-out = parallel closed form, also for T > 2M-1 and S != 2M-1."""
    g = rng(3)
    err = 0.0
    for M, S, T, L, d in ((4, 4, 16.0, 37, 5), (3, 5, 11.0, 20, 3), (5, 9, 9.0, 25, 4), (2, 2, 6.5, 19, 2)):
        q, k, v = (g.standard_normal((2, 2, L, d)) for _ in range(3))
        ref = orc.forward(q, k, v, M, S, T, form="naive")
        for form in ("modes", "parallel"):
            r = orc.forward(q, k, v, M, S, T, form=form)
            err = _worst(err, float(np.abs(r["o"] - ref["o"]).max()), float(np.abs(r["lse"] - ref["lse"]).max()))
    return err


# ------------------------------------- P6: lag form vs absolute (Alg. 1) form

def lag_vs_absolute(orc, M, S, T, L=40, d=4, seed=13):
    g = rng(seed)
    q, k, v = (g.standard_normal((1, 2, L, d)) for _ in range(3))
    a = orc.forward(q, k, v, M, S, T, form="naive")["o"]
    b = orc.forward(q, k, v, M, S, T, form="absolute")["o"]
    return float(np.linalg.norm(a - b) / np.linalg.norm(a))


def pin_absolute_bruteforce(orc):
    """Absolute form (Alg. 1, Sec. 3.2): slot j of token t holds sum_{t'<=t} D_M(t' - Delta_j) k_t',
    the Dirichlet kernel anchored at absolute phase Delta_j, here by brute force with the
    sine-ratio D_M, the grid round(j T/S) and the mask t >= Delta_j computed in this file."""
    g = rng(31)
    err = 0.0
    for M, S, T, L, d in ((3, 4, 10.0, 23, 3), (4, 6, 21.0, 40, 2), (3, 5, 5.0, 17, 4)):
        q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
        r = orc.forward(q, k, v, M, S, T, form="absolute")
        w = 2 * np.pi / T
        delta = np.round(np.arange(S) * T / S)
        for t in range(L):
            u = np.arange(t + 1)
            W = dirichlet_sine_ratio(M, w, u[None, :] - delta[:, None])   # [S, t+1]
            Ks = W @ k[0, 0, : t + 1]
            Vs = W @ v[0, 0, : t + 1]
            s = Ks @ q[0, 0, t] / np.sqrt(d)
            valid = t >= delta
            p, lse = _softmax_masked(s[None], valid[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ Vs).max()),
                      float(abs(r["lse"][0, 0, t] - lse[0])))
    return err


# ----------------------------------------------------------- P7: one mode

def pin_single_mode(orc):
    """M = 1 (one slot): D_1 = 1, so o_t = sum_{t'<=t} v_t' (Eq. dirichlet with M = 1)."""
    g = rng(17)
    q, k, v = (g.standard_normal((1, 3, 12, 4)) for _ in range(3))
    r = orc.forward(q, k, v, 1, 1, 5.0, form="naive")
    return float(np.abs(r["o"] - np.cumsum(v, axis=2)).max())


# ---------------------------------------------- P9: gradients vs differences

def pin_backward_fd(orc, h=1e-6):
    """Analytic VJP = central finite differences of the Alg. 2 forward, loss = sum(dO * O)."""
    g = rng(21)
    err = 0.0
    for M, S, T, L, d in ((3, 4, 9.0, 7, 3), (3, 5, 5.0, 12, 2)):
        q, k, v, do = (g.standard_normal((1, 1, L, d)) for _ in range(4))
        dq, dk, dv = orc.backward(q, k, v, do, M, S, T)
        for x, gx in ((q, dq), (k, dk), (v, dv)):
            fd = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                x0 = x[idx]
                x[idx] = x0 + h
                lp = float((orc.forward(q, k, v, M, S, T)["o"] * do).sum())
                x[idx] = x0 - h
                lm = float((orc.forward(q, k, v, M, S, T)["o"] * do).sum())
                x[idx] = x0
                fd[idx] = (lp - lm) / (2 * h)
            err = _worst(err, float(np.abs(fd - gx).max() / (np.abs(gx).max() + 1e-30)))
    return err


def pin_backward_fd_absolute(orc, h=1e-6):
    """The absolute form's VJP = central finite differences of its Alg. 1 forward, loss = sum(dO * O)."""
    g = rng(37)
    err = 0.0
    for M, S, T, L, d in ((3, 4, 9.0, 8, 3), (2, 3, 7.0, 11, 2)):
        q, k, v, do = (g.standard_normal((1, 1, L, d)) for _ in range(4))
        dq, dk, dv = orc.backward(q, k, v, do, M, S, T, form="absolute")
        for x, gx in ((q, dq), (k, dk), (v, dv)):
            fd = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                x0 = x[idx]
                x[idx] = x0 + h
                lp = float((orc.forward(q, k, v, M, S, T, form="absolute")["o"] * do).sum())
                x[idx] = x0 - h
                lm = float((orc.forward(q, k, v, M, S, T, form="absolute")["o"] * do).sum())
                x[idx] = x0
                fd[idx] = (lp - lm) / (2 * h)
            err = _worst(err, float(np.abs(fd - gx).max() / (np.abs(gx).max() + 1e-30)))
    return err


# ------------------------------------------------- P10: state hand-off

def pin_state_handoff(orc):
    """Prefill of L1 tokens, then the remaining tokens from the returned state with pos0 = L1,
    equals one pass over all tokens (Eq. recurrence is a one-step map)."""
    g = rng(23)
    M, S, T, L1, L2, d = 4, 5, 13.0, 11, 9, 3
    q, k, v = (g.standard_normal((1, 2, L1 + L2, d)) for _ in range(3))
    full = orc.forward(q, k, v, M, S, T, return_state=True)
    a = orc.forward(q[:, :, :L1], k[:, :, :L1], v[:, :, :L1], M, S, T, return_state=True)
    b = orc.forward(q[:, :, L1:], k[:, :, L1:], v[:, :, L1:], M, S, T, state=a["state"], pos0=L1,
                    return_state=True)
    return _worst(float(np.abs(b["o"] - full["o"][:, :, L1:]).max()),
               float(np.abs(b["state"] - full["state"]).max()),
               float(np.abs(a["o"] - full["o"][:, :, :L1]).max()))


# ------------------------------------------------- P8: state decay (Sec. 3.3)

def _latest_in_class(t, dj, T):
    """Latest token u <= t with u = dj (mod T), for integers t >= dj."""
    return int(t - ((t - dj) % T))


def pin_decay_swa(orc):
    """Sec. 3.3 at T = 2M-1: D_M(x) is 1 at x = 0 (mod 2M-1) and 0 at other integers, so the
    decay overwrites slot j with k_t whenever t = Delta_j (mod 2M-1) and leaves it alone
    otherwise.  Slot j then holds the latest token of its residue class; at S = 2M-1 the slots
    hold exactly the last 2M-1 tokens, i.e. sliding-window softmax attention, which is checked
    here against the textbook window [t-2M+2, t] as well."""
    g = rng(41)
    err = 0.0
    for M, S, L, d in ((3, 5, 23, 3), (4, 7, 30, 2), (2, 3, 2, 2), (3, 4, 19, 3), (3, 8, 21, 2)):
        T = 2 * M - 1
        q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
        r = orc.forward_decay(q, k, v, M, S, float(T))
        delta = np.round(np.arange(S) * T / S).astype(int)       # half to even, as the grid reading
        for t in range(L):
            valid = t >= delta
            rows = np.array([_latest_in_class(t, dj, T) if ok else 0 for dj, ok in zip(delta, valid)])
            s = k[0, 0, rows] @ q[0, 0, t] / np.sqrt(d)
            p, lse = _softmax_masked(s[None], valid[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ v[0, 0, rows]).max()),
                         float(abs(r["lse"][0, 0, t] - lse[0])))
            if S == T:
                win = np.arange(max(0, t - T + 1), t + 1)
                sw = k[0, 0, win] @ q[0, 0, t] / np.sqrt(d)
                pw = np.exp(sw - sw.max())
                pw /= pw.sum()
                err = _worst(err, float(np.abs(r["o"][0, 0, t] - pw @ v[0, 0, win]).max()))
    return err


def pin_decay_closed_form(orc):
    """Unrolled decay recurrence: slot j of token t holds
    sum_{u<=t} D_j(u) prod_{u<x<=t} (1 - D_j(x)) k_u with D_j(x) = D_M(x - Delta_j), evaluated
    here with the sine-ratio D_M, for periods above 2M-1 and an explicit omega."""
    g = rng(43)
    err = 0.0
    for M, S, T, om, L, d in ((3, 4, 10.0, 0.0, 17, 3), (4, 6, 21.0, 0.0, 15, 2), (2, 5, 9.0, 0.41, 13, 3)):
        q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
        r = orc.forward_decay(q, k, v, M, S, T, omega=om, return_state=True)
        w = om if om > 0 else 2 * np.pi / T
        delta = np.round(np.arange(S) * T / S)
        Dx = dirichlet_sine_ratio(M, w, np.arange(L)[None, :] - delta[:, None])   # [S, L]
        for t in range(L):
            W = np.zeros((S, t + 1))
            for u in range(t + 1):
                W[:, u] = Dx[:, u] * np.prod(1.0 - Dx[:, u + 1: t + 1], axis=1)
            Ks, Vs = W @ k[0, 0, : t + 1], W @ v[0, 0, : t + 1]
            valid = t >= delta
            p, lse = _softmax_masked((Ks @ q[0, 0, t] / np.sqrt(d))[None], valid[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ Vs).max()),
                         float(abs(r["lse"][0, 0, t] - lse[0])))
        err = _worst(err, float(np.abs(r["state"][0, 0, 0] - Ks).max()),
                     float(np.abs(r["state"][0, 0, 1] - Vs).max()))
    return err


def pin_decay_single_mode(orc):
    """M = 1: D_1 = 1 everywhere, so the decay empties every slot and refills it with the current
    token; the output is v_t itself."""
    g = rng(47)
    q, k, v = (g.standard_normal((2, 2, 11, 3)) for _ in range(3))
    r = orc.forward_decay(q, k, v, 1, 3, 7.0)
    return float(np.abs(r["o"] - v).max())


def pin_decay_handoff(orc):
    """Prefill of L1 tokens, then the rest from the returned slot state with pos0 = L1 (which sets
    both the phase of D_j and the slot mask), equals one pass."""
    g = rng(53)
    M, S, T, L1, L2, d = 3, 5, 13.0, 4, 12, 3
    q, k, v = (g.standard_normal((1, 2, L1 + L2, d)) for _ in range(3))
    full = orc.forward_decay(q, k, v, M, S, T, return_state=True)
    a = orc.forward_decay(q[:, :, :L1], k[:, :, :L1], v[:, :, :L1], M, S, T, return_state=True)
    b = orc.forward_decay(q[:, :, L1:], k[:, :, L1:], v[:, :, L1:], M, S, T, state=a["state"], pos0=L1,
                          return_state=True)
    return _worst(float(np.abs(b["o"] - full["o"][:, :, L1:]).max()),
                  float(np.abs(b["state"] - full["state"]).max()),
                  float(np.abs(a["o"] - full["o"][:, :, :L1]).max()))


def pin_decay_backward_fd(orc, h=1e-6):
    """The decayed form's VJP = central finite differences of its forward, loss = sum(dO * O), for
    T above 2M-1, at T = 2M-1 (sliding window) and from a later start position."""
    g = rng(59)
    err = 0.0
    for M, S, T, L, d, pos0 in ((3, 4, 10.0, 8, 3, 0), (2, 3, 3.0, 9, 2, 0), (2, 5, 11.0, 7, 2, 6)):
        q, k, v, do = (g.standard_normal((1, 1, L, d)) for _ in range(4))
        dq, dk, dv = orc.backward_decay(q, k, v, do, M, S, T, pos0=pos0)

        def loss():
            return float((orc.forward_decay(q, k, v, M, S, T, pos0=pos0)["o"] * do).sum())

        for x, gx in ((q, dq), (k, dk), (v, dv)):
            fd = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                x0 = x[idx]
                x[idx] = x0 + h
                lp = loss()
                x[idx] = x0 - h
                lm = loss()
                x[idx] = x0
                fd[idx] = (lp - lm) / (2 * h)
            err = _worst(err, float(np.abs(fd - gx).max() / (np.abs(gx).max() + 1e-30)))
    return err


# ------------------------------------ explicit frequency and softmax scale

def pin_explicit_omega_scale(orc):
    """An explicit mode frequency omega > 0 replaces 2 pi / T in D_M (Sec. 3.1) while the grid
    stays round(j T / S), and an explicit scale replaces 1/sqrt(d_k) (Eq. output): the lag and
    absolute forms against a sine-ratio brute force at that omega and scale."""
    g = rng(73)
    M, S, T, L, d, om, sc = 3, 4, 12.0, 15, 3, 0.37, 0.8
    q, k, v = (g.standard_normal((1, 1, L, d)) for _ in range(3))
    delta = np.round(np.arange(S) * T / S)
    err = 0.0
    for form, arg in (("naive", lambda t, u: (t - u)[None, :] - delta[:, None]),
                      ("modes", lambda t, u: (t - u)[None, :] - delta[:, None]),
                      ("absolute", lambda t, u: u[None, :] - delta[:, None])):
        r = orc.forward(q, k, v, M, S, T, omega=om, scale=sc, form=form)
        for t in range(L):
            u = np.arange(t + 1)
            W = dirichlet_sine_ratio(M, om, arg(t, u))
            Ks, Vs = W @ k[0, 0, : t + 1], W @ v[0, 0, : t + 1]
            p, lse = _softmax_masked((sc * (Ks @ q[0, 0, t]))[None], (t >= delta)[None])
            err = _worst(err, float(np.abs(r["o"][0, 0, t] - p[0] @ Vs).max()),
                         float(abs(r["lse"][0, 0, t] - lse[0])))
    return err


# ------------------------------------------------ token selection (want)

def pin_token_selection(orc):
    """Restricting the output to some tokens (``want``, used to sample long sequences) changes
    nothing else: selected tokens equal the full run, the others are NaN, and the state advances
    over every token (Eq. recurrence is applied to all of them)."""
    g = rng(71)
    M, S, T, L, d = 3, 4, 11.0, 19, 3
    q, k, v = (g.standard_normal((1, 2, L, d)) for _ in range(3))
    want = np.zeros(L, bool)
    want[[0, 5, 6, 13, L - 1]] = True
    err = 0.0
    for form in ("naive", "modes"):
        full = orc.forward(q, k, v, M, S, T, form=form, return_state=True)
        part = orc.forward(q, k, v, M, S, T, form=form, want=want, return_state=True)
        err = _worst(err, float(np.abs(part["o"][:, :, want] - full["o"][:, :, want]).max()),
                     float(np.abs(part["lse"][:, :, want] - full["lse"][:, :, want]).max()),
                     float(np.abs(part["state"] - full["state"]).max()))
        if not (np.isnan(part["o"][:, :, ~want]).all() and np.isnan(part["lse"][:, :, ~want]).all()):
            err = float("inf")
    return err


# --------------------------------------- NEXT: per-head periods (T in R^H)

def pin_per_head_period(orc):
    """Alg. 1 and Alg. 3 take one period per head: each head's grid round(j T_h / S), frequency
    2 pi / T_h and coefficients follow its own period.  Every head of a per-head run is checked
    against a brute force at its own period, computed here with the sine-ratio D_M: the lag form
    (weight D_M(t - u - Delta_j)), the absolute form (D_M(u - Delta_j)) and the decayed form (the
    unrolled product).  The periods differ per head, including T = 2M-1, so a head reading
    another head's period fails."""
    g = rng(61)
    M, S, L, d = 3, 5, 14, 3
    Ts = np.array([5.0, 13.0, 21.0])
    q, k, v = (g.standard_normal((2, 3, L, d)) for _ in range(3))
    lag = orc.forward(q, k, v, M, S, Ts, form="naive")
    ab = orc.forward(q, k, v, M, S, Ts, form="absolute")
    dec = orc.forward_decay(q, k, v, M, S, Ts)
    err = 0.0
    for h, T in enumerate(Ts):
        w = 2 * np.pi / T
        delta = np.round(np.arange(S) * T / S)
        Dabs = dirichlet_sine_ratio(M, w, np.arange(L)[None, :] - delta[:, None])   # D_j(u), [S, L]
        for b in range(2):
            for t in range(L):
                u = np.arange(t + 1)
                Wd = np.zeros((S, t + 1))
                for uu in range(t + 1):
                    Wd[:, uu] = Dabs[:, uu] * np.prod(1.0 - Dabs[:, uu + 1: t + 1], axis=1)
                for r, W in ((lag, dirichlet_sine_ratio(M, w, (t - u)[None, :] - delta[:, None])),
                             (ab, Dabs[:, : t + 1]), (dec, Wd)):
                    Ks, Vs = W @ k[b, h, : t + 1], W @ v[b, h, : t + 1]
                    p, lse = _softmax_masked((Ks @ q[b, h, t] / np.sqrt(d))[None], (t >= delta)[None])
                    err = _worst(err, float(np.abs(r["o"][b, h, t] - p[0] @ Vs).max()),
                                 float(abs(r["lse"][b, h, t] - lse[0])))
    return err


def pin_per_head_period_backward(orc, h=1e-6):
    """The VJPs with per-head periods (lag, absolute and decayed forms) = central differences of
    the per-head forwards."""
    g = rng(67)
    M, S, L, d = 2, 3, 6, 2
    Ts = np.array([3.0, 8.0])
    q, k, v, do = (g.standard_normal((1, 2, L, d)) for _ in range(4))
    err = 0.0
    for fwd, bwd in ((lambda: orc.forward(q, k, v, M, S, Ts, form="parallel")["o"],
                      lambda: orc.backward(q, k, v, do, M, S, Ts)),
                     (lambda: orc.forward(q, k, v, M, S, Ts, form="absolute")["o"],
                      lambda: orc.backward(q, k, v, do, M, S, Ts, form="absolute")),
                     (lambda: orc.forward_decay(q, k, v, M, S, Ts)["o"],
                      lambda: orc.backward_decay(q, k, v, do, M, S, Ts))):
        grads = bwd()
        for x, gx in zip((q, k, v), grads):
            fd = np.zeros_like(x)
            for idx in np.ndindex(x.shape):
                x0 = x[idx]
                x[idx] = x0 + h
                lp = float((fwd() * do).sum())
                x[idx] = x0 - h
                lm = float((fwd() * do).sum())
                x[idx] = x0
                fd[idx] = (lp - lm) / (2 * h)
            err = _worst(err, float(np.abs(fd - gx).max() / (np.abs(gx).max() + 1e-30)))
    return err


ALL_PINS = {
    "dirichlet_identity": (pin_dirichlet_identity, 1e-12),
    "dirichlet_samples": (pin_dirichlet_samples, 1e-13),
    "grid": (pin_grid, 0.0),
    "translated_coefficients": (pin_translated_coefficients, 1e-12),
    "state_closed_form": (pin_state_closed_form, 1e-11),
    "causal_attention": (pin_causal_attention, 1e-12),
    "aliasing": (pin_aliasing, 1e-11),
    "blurry_bruteforce": (pin_blurry_bruteforce, 1e-11),
    "forms_agree": (pin_forms_agree, 1e-11),
    "single_mode": (pin_single_mode, 1e-12),
    "backward_fd": (pin_backward_fd, 1e-6),
    "absolute_bruteforce": (pin_absolute_bruteforce, 1e-11),
    "backward_fd_absolute": (pin_backward_fd_absolute, 1e-6),
    "state_handoff": (pin_state_handoff, 1e-12),
    "decay_swa": (pin_decay_swa, 1e-12),
    "decay_closed_form": (pin_decay_closed_form, 1e-11),
    "decay_single_mode": (pin_decay_single_mode, 1e-13),
    "decay_handoff": (pin_decay_handoff, 1e-12),
    "decay_backward_fd": (pin_decay_backward_fd, 1e-6),
    "per_head_period": (pin_per_head_period, 1e-11),
    "token_selection": (pin_token_selection, 0.0),
    "explicit_omega_scale": (pin_explicit_omega_scale, 1e-11),
    "per_head_period_backward": (pin_per_head_period_backward, 1e-6),
}
