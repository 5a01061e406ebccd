/*
 * bla_oracle.c -- float64 CPU oracle for Blurry Window Attention (BLA), lag form.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct reference
 * that the CUDA path is checked against.  Only tests/, __graft_entry__.smoke()
 * and bench.py's cpu_baseline leg may load it.  It shares no code, header,
 * table or constant with the CUDA library and includes nothing from it.
 *
 * Notation follows the paper (arxiv 2606.09862, "Blurry Window Attention"):
 *   M        number of Fourier modes, m = 0..M-1
 *   T        period; clamped T <- max(T, 2M-1) as in Alg. 1 and Alg. 3
 *   omega    fundamental frequency, 2*pi/T unless given explicitly (Sec. 3.1)
 *   S        number of slots; the paper always has S = 2M-1 (Table 1)
 *   Delta_j  dilated time grid, round(j*T/S), j = 0..S-1 (Alg. 1-3 "dilated_time",
 *            generalised from S = 2M-1 to any S; equal to the paper's grid at S = 2M-1)
 *   A, B     Fourier coefficients of the translated Dirichlet kernels, Eq. (translated):
 *            A[j,0] = 1/(2M-1), A[j,m>0] = 2 cos(m w Delta_j)/(2M-1),
 *            B[j,0] = 0,        B[j,m>0] = 2 sin(m w Delta_j)/(2M-1)
 *
 * State layout used on this interface (per batch-head, doubles):
 *   [2 (K then V)][M][2 (cos, sin)][d]     -- the sin row of mode 0 is always 0.
 *
 * Forms provided (all float64):
 *   orc_forward_naive     Alg. 2 ("Naive recurrent BLA") written out: rotate the
 *                         mode state (Eq. recurrence), rebuild the slots
 *                         (Eq. compressed), masked softmax over slots (Eq. output).
 *   orc_forward_modes     the same recurrence, but the slot read-out uses the
 *                         exchange of the sums over slots and over modes that the
 *                         paper makes in Eq. (conv): q.K~[j] = sum_m A[j,m] (q.Kcos[m])
 *                         + B[j,m] (q.Ksin[m]).  Exact rearrangement, pinned to the
 *                         naive form by the tests.
 *   orc_forward_parallel  closed form of the states, Eq. (states), combined with the
 *                         translated Dirichlet kernel, Eq. (translated_dirichelt):
 *                         K~_t[j] = sum_{t'<=t} D_M(t - t' - Delta_j) k_t'.
 *   orc_forward_absolute  Alg. 1 ("Efficient recurrent BLA"), the time-rolling
 *                         cumulative-sum form of Sec. 3.2 (pins only).
 *   orc_forward_decay     Alg. 1 with the state decay of Sec. 3.3: the previous
 *                         slot state is multiplied by (1 - D_j(t)) before the token
 *                         is added with weight D_j(t) (slot-space state [S][d]).
 *   orc_backward_decay    its vector-Jacobian product: the chain rule below with the
 *                         unrolled decay weight D_j(u) prod_{u<x<=t} (1 - D_j(x)) (pinned
 *                         to finite differences of orc_forward_decay).
 *   orc_backward_parallel vector-Jacobian product of the parallel form, written out
 *                         by the chain rule (no paper counterpart; pinned to central
 *                         finite differences of orc_forward_naive by the tests).
 *                         With form 3 it is the VJP of the absolute form instead: the
 *                         same chain rule with the weight D_M(t' - Delta_j) of Alg. 1's
 *                         "interpolate" in place of D_M(t - t' - Delta_j) (pinned to
 *                         finite differences of orc_forward_absolute).
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#define ORC_PI 3.14159265358979323846

typedef struct {
    int L, dk, dv, M, S;
    double T;        /* effective (clamped) period */
    double w;        /* omega */
    double scale;    /* softmax scale */
    long long pos0;  /* absolute index of token 0 (for the slot mask) */
} orc_cfg;

/* Alg. 1 / Alg. 3: "Clamp period: T <- max(T, 2M-1)". */
double orc_period(int M, double T)
{
    double r = 2.0 * M - 1.0;
    return T < r ? r : T;
}

/* Sec. 3.1: omega = 2*pi/T; an explicit omega > 0 overrides it. */
double orc_omega(int M, double T, double omega)
{
    return omega > 0.0 ? omega : 2.0 * ORC_PI / orc_period(M, T);
}

/* Dilated time grid: round(j*T/S), round half to even (nearbyint in the
 * default rounding mode). */
void orc_delta(int M, int S, double T, double *delta)
{
    double Te = orc_period(M, T);
    for (int j = 0; j < S; ++j) delta[j] = nearbyint((double)j * Te / (double)S);
}

/* Eq. (translated): A, B in R^{S x M}. */
void orc_tables(int M, int S, double T, double omega, double *delta, double *A, double *B)
{
    double w = orc_omega(M, T, omega);
    double n = 2.0 * M - 1.0;
    orc_delta(M, S, T, delta);
    for (int j = 0; j < S; ++j) {
        A[j * M + 0] = 1.0 / n;
        B[j * M + 0] = 0.0;
        for (int m = 1; m < M; ++m) {
            A[j * M + m] = 2.0 * cos(m * w * delta[j]) / n;
            B[j * M + m] = 2.0 * sin(m * w * delta[j]) / n;
        }
    }
}

/* Eq. (dirichlet) with a general omega: D_M(x) = 1/(2M-1) + 2/(2M-1) sum_{m>=1} cos(m w x). */
double orc_dirichlet(int M, double w, double x)
{
    double n = 2.0 * M - 1.0;
    double acc = 1.0 / n;
    for (int m = 1; m < M; ++m) acc += 2.0 / n * cos(m * w * x);
    return acc;
}

/* ---------------------------------------------------------------- helpers */

static void load_state(const orc_cfg *c, const double *st, double *Kc, double *Ks, double *Vc, double *Vs)
{
    int M = c->M, dk = c->dk, dv = c->dv;
    if (!st) {
        memset(Kc, 0, sizeof(double) * M * dk); memset(Ks, 0, sizeof(double) * M * dk);
        memset(Vc, 0, sizeof(double) * M * dv); memset(Vs, 0, sizeof(double) * M * dv);
        return;
    }
    const double *sk = st, *sv = st + (size_t)2 * M * dk;
    for (int m = 0; m < M; ++m) {
        memcpy(Kc + m * dk, sk + (size_t)(2 * m) * dk, sizeof(double) * dk);
        memcpy(Ks + m * dk, sk + (size_t)(2 * m + 1) * dk, sizeof(double) * dk);
        memcpy(Vc + m * dv, sv + (size_t)(2 * m) * dv, sizeof(double) * dv);
        memcpy(Vs + m * dv, sv + (size_t)(2 * m + 1) * dv, sizeof(double) * dv);
    }
}

static void store_state(const orc_cfg *c, double *st, const double *Kc, const double *Ks, const double *Vc, const double *Vs)
{
    int M = c->M, dk = c->dk, dv = c->dv;
    double *sk = st, *sv = st + (size_t)2 * M * dk;
    for (int m = 0; m < M; ++m) {
        memcpy(sk + (size_t)(2 * m) * dk, Kc + m * dk, sizeof(double) * dk);
        memcpy(sk + (size_t)(2 * m + 1) * dk, Ks + m * dk, sizeof(double) * dk);
        memcpy(sv + (size_t)(2 * m) * dv, Vc + m * dv, sizeof(double) * dv);
        memcpy(sv + (size_t)(2 * m + 1) * dv, Vs + m * dv, sizeof(double) * dv);
    }
}

/* Eq. (recurrence), applied to one d-vector state (Xc, Xs) with input x:
 *   Xc[m] <- cos(m w) Xc[m] - sin(m w) Xs[m] + x
 *   Xs[m] <- sin(m w) Xc[m] + cos(m w) Xs[m]
 * (right-hand sides use the values before the update, as in the equation). */
static void rotate_add(int M, int d, double w, double *Xc, double *Xs, const double *x)
{
    for (int m = 0; m < M; ++m) {
        double cw = cos(m * w), sw = sin(m * w);
        double *xc = Xc + (size_t)m * d, *xs = Xs + (size_t)m * d;
        for (int i = 0; i < d; ++i) {
            double a = xc[i], b = xs[i];
            xc[i] = cw * a - sw * b + x[i];
            xs[i] = sw * a + cw * b;
        }
    }
}

/* Masked softmax over slots (Eq. output; mask "t >= dilated_time").  Writes p
 * (0 on masked slots) and returns log-sum-exp of the unmasked scores. */
static double masked_softmax(int S, const double *s, const double *delta, long long tabs, double *p)
{
    double mx = -INFINITY;
    for (int j = 0; j < S; ++j)
        if ((double)tabs >= delta[j] && s[j] > mx) mx = s[j];
    double sum = 0.0;
    for (int j = 0; j < S; ++j) {
        p[j] = ((double)tabs >= delta[j]) ? exp(s[j] - mx) : 0.0;
        sum += p[j];
    }
    for (int j = 0; j < S; ++j) p[j] /= sum;
    return mx + log(sum);
}

/* ------------------------------------------------ Alg. 2, written out */

static void head_naive(const orc_cfg *c, const double *A, const double *B, const double *delta,
                       const double *q, const double *k, const double *v,
                       double *o, double *lse, double *st, const unsigned char *want)
{
    int M = c->M, S = c->S, dk = c->dk, dv = c->dv;
    double *Kc = malloc(sizeof(double) * M * dk), *Ks = malloc(sizeof(double) * M * dk);
    double *Vc = malloc(sizeof(double) * M * dv), *Vs = malloc(sizeof(double) * M * dv);
    double *Kt = malloc(sizeof(double) * S * dk), *Vt = malloc(sizeof(double) * S * dv);
    double *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S);
    load_state(c, st, Kc, Ks, Vc, Vs);
    for (int t = 0; t < c->L; ++t) {
        /* "Update the KV state" */
        rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)t * dk);
        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);
        if (want && !want[t]) continue;
        /* "Compute interpolated keys and values": K~ = A.Kcos + B.Ksin, Eq. (compressed) */
        for (int j = 0; j < S; ++j) {
            for (int i = 0; i < dk; ++i) {
                double acc = 0.0;
                for (int m = 0; m < M; ++m) acc += A[j * M + m] * Kc[m * dk + i] + B[j * M + m] * Ks[m * dk + i];
                Kt[j * dk + i] = acc;
            }
            for (int i = 0; i < dv; ++i) {
                double acc = 0.0;
                for (int m = 0; m < M; ++m) acc += A[j * M + m] * Vc[m * dv + i] + B[j * M + m] * Vs[m * dv + i];
                Vt[j * dv + i] = acc;
            }
        }
        /* "Update output": softmax(q.K~^T * scale + M_BLA) . V~, Eq. (output) */
        const double *qt = q + (size_t)t * dk;
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int i = 0; i < dk; ++i) acc += qt[i] * Kt[j * dk + i];
            s[j] = c->scale * acc;
        }
        double l = masked_softmax(S, s, delta, c->pos0 + t, p);
        if (lse) lse[t] = l;
        double *ot = o + (size_t)t * dv;
        for (int i = 0; i < dv; ++i) {
            double acc = 0.0;
            for (int j = 0; j < S; ++j) acc += p[j] * Vt[j * dv + i];
            ot[i] = acc;
        }
    }
    if (st) store_state(c, st, Kc, Ks, Vc, Vs);
    free(Kc); free(Ks); free(Vc); free(Vs); free(Kt); free(Vt); free(s); free(p);
}

/* ------------------------------- same recurrence, read-out through the modes */

static void head_modes(const orc_cfg *c, const double *A, const double *B, const double *delta,
                       const double *q, const double *k, const double *v,
                       double *o, double *lse, double *st, const unsigned char *want)
{
    int M = c->M, S = c->S, dk = c->dk, dv = c->dv;
    double *Kc = malloc(sizeof(double) * M * dk), *Ks = malloc(sizeof(double) * M * dk);
    double *Vc = malloc(sizeof(double) * M * dv), *Vs = malloc(sizeof(double) * M * dv);
    double *yc = malloc(sizeof(double) * M), *ys = malloc(sizeof(double) * M);
    double *uc = malloc(sizeof(double) * M), *us = malloc(sizeof(double) * M);
    double *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S);
    load_state(c, st, Kc, Ks, Vc, Vs);
    for (int t = 0; t < c->L; ++t) {
        rotate_add(M, dk, c->w, Kc, Ks, k + (size_t)t * dk);
        rotate_add(M, dv, c->w, Vc, Vs, v + (size_t)t * dv);
        if (want && !want[t]) continue;
        const double *qt = q + (size_t)t * dk;
        /* q.Kcos[m], q.Ksin[m] */
        for (int m = 0; m < M; ++m) {
            double a = 0.0, b = 0.0;
            for (int i = 0; i < dk; ++i) { a += qt[i] * Kc[m * dk + i]; b += qt[i] * Ks[m * dk + i]; }
            yc[m] = a; ys[m] = b;
        }
        /* s_j = scale * sum_m (A[j,m] q.Kcos[m] + B[j,m] q.Ksin[m]) */
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) acc += A[j * M + m] * yc[m] + B[j * M + m] * ys[m];
            s[j] = c->scale * acc;
        }
        double l = masked_softmax(S, s, delta, c->pos0 + t, p);
        if (lse) lse[t] = l;
        /* o = sum_j p_j V~[j] = sum_m (sum_j p_j A[j,m]) Vcos[m] + (sum_j p_j B[j,m]) Vsin[m] */
        for (int m = 0; m < M; ++m) {
            double a = 0.0, b = 0.0;
            for (int j = 0; j < S; ++j) { a += p[j] * A[j * M + m]; b += p[j] * B[j * M + m]; }
            uc[m] = a; us[m] = b;
        }
        double *ot = o + (size_t)t * dv;
        for (int i = 0; i < dv; ++i) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) acc += uc[m] * Vc[m * dv + i] + us[m] * Vs[m * dv + i];
            ot[i] = acc;
        }
    }
    if (st) store_state(c, st, Kc, Ks, Vc, Vs);
    free(Kc); free(Ks); free(Vc); free(Vs); free(yc); free(ys); free(uc); free(us); free(s); free(p);
}

/* ------------------------------------------ parallel ("blurry mask") form */

/* D_M(y) for every integer y in [-(Dmax), L-1], where Dmax = max_j Delta_j. */
static double *dirichlet_table(const orc_cfg *c, const double *delta, int *off)
{
    int dmax = 0;
    for (int j = 0; j < c->S; ++j) if ((int)delta[j] > dmax) dmax = (int)delta[j];
    int n = c->L + dmax;
    double *tab = malloc(sizeof(double) * (n > 0 ? n : 1));
    for (int y = -dmax; y < c->L; ++y) tab[y + dmax] = orc_dirichlet(c->M, c->w, (double)y);
    *off = dmax;
    return tab;
}

static void head_parallel(const orc_cfg *c, const double *delta,
                          const double *q, const double *k, const double *v, double *o, double *lse)
{
    int S = c->S, dk = c->dk, dv = c->dv, L = c->L, off;
    double *Dt = dirichlet_table(c, delta, &off);
    double *qk = malloc(sizeof(double) * (L > 0 ? L : 1));
    double *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S);
    for (int t = 0; t < L; ++t) {
        const double *qt = q + (size_t)t * dk;
        for (int u = 0; u <= t; ++u) {
            double acc = 0.0;
            for (int i = 0; i < dk; ++i) acc += qt[i] * k[(size_t)u * dk + i];
            qk[u] = acc;
        }
        /* s[t,j] = scale * sum_{t'<=t} D_M(t - t' - Delta_j) (q_t . k_t') */
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int u = 0; u <= t; ++u) acc += Dt[t - u - (int)delta[j] + off] * qk[u];
            s[j] = c->scale * acc;
        }
        double l = masked_softmax(S, s, delta, c->pos0 + t, p);
        if (lse) lse[t] = l;
        /* o_t = sum_j p_j sum_{t'<=t} D_M(t - t' - Delta_j) v_t' */
        double *ot = o + (size_t)t * dv;
        for (int i = 0; i < dv; ++i) ot[i] = 0.0;
        for (int u = 0; u <= t; ++u) {
            double g = 0.0;
            for (int j = 0; j < S; ++j) g += p[j] * Dt[t - u - (int)delta[j] + off];
            for (int i = 0; i < dv; ++i) ot[i] += g * v[(size_t)u * dv + i];
        }
    }
    free(Dt); free(qk); free(s); free(p);
}

/* -------------------------------------------- Alg. 1, absolute time frame */

static void head_absolute(const orc_cfg *c, const double *A, const double *B, const double *delta,
                          const double *q, const double *k, const double *v, double *o, double *lse)
{
    int M = c->M, S = c->S, dk = c->dk, dv = c->dv;
    double *Kp = calloc((size_t)S * dk, sizeof(double)), *Vp = calloc((size_t)S * dv, sizeof(double));
    double *ip = malloc(sizeof(double) * S), *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S);
    for (int t = 0; t < c->L; ++t) {
        /* interpolate = cos(t.modes) A^T + sin(t.modes) B^T, Eq. (compressed_simplified) */
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) acc += cos(t * m * c->w) * A[j * M + m] + sin(t * m * c->w) * B[j * M + m];
            ip[j] = acc;
        }
        /* K_prev <- K_prev + K[t] (x) interpolate */
        for (int j = 0; j < S; ++j) {
            for (int i = 0; i < dk; ++i) Kp[j * dk + i] += k[(size_t)t * dk + i] * ip[j];
            for (int i = 0; i < dv; ++i) Vp[j * dv + i] += v[(size_t)t * dv + i] * ip[j];
        }
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int i = 0; i < dk; ++i) acc += q[(size_t)t * dk + i] * Kp[j * dk + i];
            s[j] = c->scale * acc;
        }
        double l = masked_softmax(S, s, delta, c->pos0 + t, p);
        if (lse) lse[t] = l;
        for (int i = 0; i < dv; ++i) {
            double acc = 0.0;
            for (int j = 0; j < S; ++j) acc += p[j] * Vp[j * dv + i];
            o[(size_t)t * dv + i] = acc;
        }
    }
    free(Kp); free(Vp); free(ip); free(s); free(p);
}

/* ------------------------------------------- Sec. 3.3: Alg. 1 with state decay
 *
 * The slot-space state of Alg. 1, where the previous state is multiplied by (1 - D_j(t))
 * before the token's key (value) is added with Alg. 1's weight D_j(t):
 *     K~[j] <- (1 - D_j(t)) K~[j] + D_j(t) k_t,      V~[j] likewise,
 * D_j(t) = "interpolate"[j] = cos(t.modes) A^T + sin(t.modes) B^T (Eq. compressed_simplified)
 * at the absolute token index t = pos0 + i.  Read-out as in Alg. 1: masked softmax of
 * scale q_t . K~[j] over the slots, output sum_j p_j V~[j].
 * State (per head, in/out, may be NULL for a zero start): [S][dk] then [S][dv].
 */
static void head_decay(const orc_cfg *c, const double *A, const double *B, const double *delta,
                       const double *q, const double *k, const double *v, double *o, double *lse, double *st)
{
    int M = c->M, S = c->S, dk = c->dk, dv = c->dv;
    double *own = st ? NULL : calloc((size_t)S * (dk + dv), sizeof(double));
    double *Kp = st ? st : own, *Vp = Kp + (size_t)S * dk;
    double *ip = malloc(sizeof(double) * S), *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S);
    for (int i = 0; i < c->L; ++i) {
        double t = (double)(c->pos0 + i);
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) acc += cos(t * m * c->w) * A[j * M + m] + sin(t * m * c->w) * B[j * M + m];
            ip[j] = acc;
        }
        for (int j = 0; j < S; ++j) {
            double keep = 1.0 - ip[j];
            for (int e = 0; e < dk; ++e) Kp[j * dk + e] = keep * Kp[j * dk + e] + ip[j] * k[(size_t)i * dk + e];
            for (int e = 0; e < dv; ++e) Vp[j * dv + e] = keep * Vp[j * dv + e] + ip[j] * v[(size_t)i * dv + e];
        }
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int e = 0; e < dk; ++e) acc += q[(size_t)i * dk + e] * Kp[j * dk + e];
            s[j] = c->scale * acc;
        }
        double l = masked_softmax(S, s, delta, c->pos0 + i, p);
        if (lse) lse[i] = l;
        for (int e = 0; e < dv; ++e) {
            double acc = 0.0;
            for (int j = 0; j < S; ++j) acc += p[j] * Vp[j * dv + e];
            o[(size_t)i * dv + e] = acc;
        }
    }
    free(own); free(ip); free(s); free(p);
}

/* ------------------------------------ VJP of the parallel form (chain rule)
 *
 *   W[t,t',j] = D_M(t - t' - Delta_j)            (t' <= t; absolute form: D_M(t' - Delta_j))
 *   s[t,j]    = scale sum_t' W (q_t . k_t'),     p = masked softmax_j(s)
 *   G[t,t']   = sum_j p[t,j] W[t,t',j],          o_t = sum_t' G[t,t'] v_t'
 * Given do:
 *   dp[t,j]   = sum_t' W[t,t',j] (do_t . v_t')
 *   ds[t,j]   = p[t,j] (dp[t,j] - sum_i p[t,i] dp[t,i])
 *   dP[t,t']  = scale sum_j ds[t,j] W[t,t',j]
 *   dq_t = sum_t' dP[t,t'] k_t',  dk_t' = sum_t dP[t,t'] q_t,  dv_t' = sum_t G[t,t'] do_t
 */
/* Index of D_M in the weight W[t,t',j]: lag form t - t' - Delta_j, absolute form t' - Delta_j. */
static int weight_arg(int absolute, int t, int u, int dj)
{
    return absolute ? u - dj : t - u - dj;
}

static void head_backward(const orc_cfg *c, const double *delta, int absolute,
                          const double *q, const double *k, const double *v, const double *dout,
                          double *dq, double *dk_, double *dv_)
{
    int S = c->S, dk = c->dk, dv = c->dv, L = c->L, off;
    double *Dt = dirichlet_table(c, delta, &off);
    double *qk = malloc(sizeof(double) * (L > 0 ? L : 1)), *dov = malloc(sizeof(double) * (L > 0 ? L : 1));
    double *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S), *dp = malloc(sizeof(double) * S);
    memset(dq, 0, sizeof(double) * (size_t)L * dk);
    memset(dk_, 0, sizeof(double) * (size_t)L * dk);
    memset(dv_, 0, sizeof(double) * (size_t)L * dv);
    for (int t = 0; t < L; ++t) {
        const double *qt = q + (size_t)t * dk, *dot = dout + (size_t)t * dv;
        for (int u = 0; u <= t; ++u) {
            double a = 0.0, b = 0.0;
            for (int i = 0; i < dk; ++i) a += qt[i] * k[(size_t)u * dk + i];
            for (int i = 0; i < dv; ++i) b += dot[i] * v[(size_t)u * dv + i];
            qk[u] = a; dov[u] = b;
        }
        for (int j = 0; j < S; ++j) {
            double a = 0.0, b = 0.0;
            for (int u = 0; u <= t; ++u) {
                double wgt = Dt[weight_arg(absolute, t, u, (int)delta[j]) + off];
                a += wgt * qk[u]; b += wgt * dov[u];
            }
            s[j] = c->scale * a; dp[j] = b;
        }
        masked_softmax(S, s, delta, c->pos0 + t, p);
        double pdp = 0.0;
        for (int j = 0; j < S; ++j) pdp += p[j] * dp[j];
        for (int u = 0; u <= t; ++u) {
            double g = 0.0, dP = 0.0;
            for (int j = 0; j < S; ++j) {
                double wgt = Dt[weight_arg(absolute, t, u, (int)delta[j]) + off];
                g += p[j] * wgt;
                dP += p[j] * (dp[j] - pdp) * wgt;
            }
            dP *= c->scale;
            for (int i = 0; i < dk; ++i) {
                dq[(size_t)t * dk + i] += dP * k[(size_t)u * dk + i];
                dk_[(size_t)u * dk + i] += dP * qt[i];
            }
            for (int i = 0; i < dv; ++i) dv_[(size_t)u * dv + i] += g * dot[i];
        }
    }
    free(Dt); free(qk); free(dov); free(s); free(p); free(dp);
}

/* ------------------------------------------- VJP of the decayed form (Sec. 3.3)
 *
 * Unrolled, the decayed slot state is a fixed linear map of the past tokens:
 *     K~_t[j] = sum_{u<=t} Wd[t,u,j] k_u,     Wd[t,u,j] = D_j(u) prod_{u<x<=t} (1 - D_j(x)),
 * with D_j(x) Alg. 1's "interpolate" at the absolute index pos0 + x (V~ likewise).  With Wd in
 * place of the weight W, the chain rule written out above head_backward applies as it stands
 * (zero initial state).
 */
static void head_backward_decay(const orc_cfg *c, const double *A, const double *B, const double *delta,
                                const double *q, const double *k, const double *v, const double *dout,
                                double *dq, double *dk_, double *dv_)
{
    int M = c->M, S = c->S, dk = c->dk, dv = c->dv, L = c->L;
    size_t nls = (size_t)(L > 0 ? L : 1) * S;
    double *ip = malloc(sizeof(double) * nls), *Wt = malloc(sizeof(double) * nls);
    double *qk = malloc(sizeof(double) * (L > 0 ? L : 1)), *dov = malloc(sizeof(double) * (L > 0 ? L : 1));
    double *s = malloc(sizeof(double) * S), *p = malloc(sizeof(double) * S), *dp = malloc(sizeof(double) * S);
    memset(dq, 0, sizeof(double) * (size_t)L * dk);
    memset(dk_, 0, sizeof(double) * (size_t)L * dk);
    memset(dv_, 0, sizeof(double) * (size_t)L * dv);
    for (int x = 0; x < L; ++x) {
        double tx = (double)(c->pos0 + x);
        for (int j = 0; j < S; ++j) {
            double acc = 0.0;
            for (int m = 0; m < M; ++m) acc += cos(tx * m * c->w) * A[j * M + m] + sin(tx * m * c->w) * B[j * M + m];
            ip[(size_t)x * S + j] = acc;
        }
    }
    for (int t = 0; t < L; ++t) {
        const double *qt = q + (size_t)t * dk, *dot = dout + (size_t)t * dv;
        for (int j = 0; j < S; ++j) {          /* Wd[t,u,j] for u = t down to 0 */
            double prod = 1.0;
            for (int u = t; u >= 0; --u) {
                Wt[(size_t)u * S + j] = ip[(size_t)u * S + j] * prod;
                prod *= 1.0 - ip[(size_t)u * S + j];
            }
        }
        for (int u = 0; u <= t; ++u) {
            double a = 0.0, b = 0.0;
            for (int i = 0; i < dk; ++i) a += qt[i] * k[(size_t)u * dk + i];
            for (int i = 0; i < dv; ++i) b += dot[i] * v[(size_t)u * dv + i];
            qk[u] = a; dov[u] = b;
        }
        for (int j = 0; j < S; ++j) {
            double a = 0.0, b = 0.0;
            for (int u = 0; u <= t; ++u) {
                a += Wt[(size_t)u * S + j] * qk[u];
                b += Wt[(size_t)u * S + j] * dov[u];
            }
            s[j] = c->scale * a; dp[j] = b;
        }
        masked_softmax(S, s, delta, c->pos0 + t, p);
        double pdp = 0.0;
        for (int j = 0; j < S; ++j) pdp += p[j] * dp[j];
        for (int u = 0; u <= t; ++u) {
            double g = 0.0, dP = 0.0;
            for (int j = 0; j < S; ++j) {
                double wgt = Wt[(size_t)u * S + j];
                g += p[j] * wgt;
                dP += p[j] * (dp[j] - pdp) * wgt;
            }
            dP *= c->scale;
            for (int i = 0; i < dk; ++i) {
                dq[(size_t)t * dk + i] += dP * k[(size_t)u * dk + i];
                dk_[(size_t)u * dk + i] += dP * qt[i];
            }
            for (int i = 0; i < dv; ++i) dv_[(size_t)u * dv + i] += g * dot[i];
        }
    }
    free(ip); free(Wt); free(qk); free(dov); free(s); free(p); free(dp);
}

/* ------------------------------------------------------------ entry points
 * Arrays are [NH][L][d] with NH = batch*heads, contiguous; state is
 * [NH][2][M][2][d] (see header).  `want` (length L, may be NULL) selects the
 * tokens whose output is computed; the state always advances over all L tokens.
 * Heads run in parallel over OpenMP threads.
 */

static orc_cfg make_cfg(int L, int dk, int dv, int M, int S, double T, double omega, double scale, long long pos0)
{
    orc_cfg c;
    c.L = L; c.dk = dk; c.dv = dv; c.M = M; c.S = S;
    c.T = orc_period(M, T);
    c.w = orc_omega(M, T, omega);
    c.scale = scale > 0.0 ? scale : 1.0 / sqrt((double)dk);
    c.pos0 = pos0;
    return c;
}

int orc_forward(int form, int NH, int L, int dk, int dv, int M, int S, double T, double omega,
                double scale, long long pos0, const double *q, const double *k, const double *v,
                double *o, double *lse, double *state, const unsigned char *want)
{
    if (NH < 0 || L < 0 || dk < 1 || dv < 1 || M < 1 || S < 1) return 1;
    orc_cfg c = make_cfg(L, dk, dv, M, S, T, omega, scale, pos0);
    double *delta = malloc(sizeof(double) * S), *A = malloc(sizeof(double) * S * M), *B = malloc(sizeof(double) * S * M);
    orc_tables(M, S, T, omega, delta, A, B);
    int nthr_stateful = (form == 0 || form == 1);
    if (!nthr_stateful && (state || pos0 != 0)) { free(delta); free(A); free(B); return 2; }
    #pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < NH; ++h) {
        const double *qh = q + (size_t)h * L * dk, *kh = k + (size_t)h * L * dk, *vh = v + (size_t)h * L * dv;
        double *oh = o + (size_t)h * L * dv, *lh = lse ? lse + (size_t)h * L : NULL;
        double *sh = state ? state + (size_t)h * 2 * M * (dk + dv) : NULL;
        switch (form) {
        case 0: head_naive(&c, A, B, delta, qh, kh, vh, oh, lh, sh, want); break;
        case 1: head_modes(&c, A, B, delta, qh, kh, vh, oh, lh, sh, want); break;
        case 2: head_parallel(&c, delta, qh, kh, vh, oh, lh); break;
        case 3: head_absolute(&c, A, B, delta, qh, kh, vh, oh, lh); break;
        default: break;
        }
    }
    free(delta); free(A); free(B);
    return (form >= 0 && form <= 3) ? 0 : 3;
}

/* Alg. 1 with the state decay of Sec. 3.3.  State is [NH][S*(dk+dv)] (slot-space K~ then
 * V~), in/out; NULL starts from zero and keeps nothing.  pos0 is the absolute index of
 * token 0 (it sets both the phase of "interpolate" and the slot mask). */
int orc_forward_decay(int NH, int L, int dk, int dv, int M, int S, double T, double omega, double scale,
                      long long pos0, const double *q, const double *k, const double *v,
                      double *o, double *lse, double *state)
{
    if (NH < 0 || L < 0 || dk < 1 || dv < 1 || M < 1 || S < 1 || pos0 < 0) return 1;
    orc_cfg c = make_cfg(L, dk, dv, M, S, T, omega, scale, pos0);
    double *delta = malloc(sizeof(double) * S), *A = malloc(sizeof(double) * S * M), *B = malloc(sizeof(double) * S * M);
    orc_tables(M, S, T, omega, delta, A, B);
    #pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < NH; ++h) {
        size_t ok = (size_t)h * L * dk, ov = (size_t)h * L * dv;
        head_decay(&c, A, B, delta, q + ok, k + ok, v + ov, o + ov, lse ? lse + (size_t)h * L : NULL,
                   state ? state + (size_t)h * S * (dk + dv) : NULL);
    }
    free(delta); free(A); free(B);
    return 0;
}

/* VJP of orc_forward_decay from the zero state, tokens at absolute indices pos0 .. pos0+L-1. */
int orc_backward_decay(int NH, int L, int dk, int dv, int M, int S, double T, double omega, double scale,
                       long long pos0, const double *q, const double *k, const double *v, const double *dout,
                       double *dq, double *dk_, double *dv_)
{
    if (NH < 0 || L < 0 || dk < 1 || dv < 1 || M < 1 || S < 1 || pos0 < 0) return 1;
    orc_cfg c = make_cfg(L, dk, dv, M, S, T, omega, scale, pos0);
    double *delta = malloc(sizeof(double) * S), *A = malloc(sizeof(double) * S * M), *B = malloc(sizeof(double) * S * M);
    orc_tables(M, S, T, omega, delta, A, B);
    #pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < NH; ++h) {
        size_t ok = (size_t)h * L * dk, ov = (size_t)h * L * dv;
        head_backward_decay(&c, A, B, delta, q + ok, k + ok, v + ov, dout + ov, dq + ok, dk_ + ok, dv_ + ov);
    }
    free(delta); free(A); free(B);
    return 0;
}

int orc_backward(int form, int NH, int L, int dk, int dv, int M, int S, double T, double omega, double scale,
                 const double *q, const double *k, const double *v, const double *dout,
                 double *dq, double *dk_, double *dv_)
{
    if (NH < 0 || L < 0 || dk < 1 || dv < 1 || M < 1 || S < 1) return 1;
    if (form != 2 && form != 3) return 3;
    orc_cfg c = make_cfg(L, dk, dv, M, S, T, omega, scale, 0);
    double *delta = malloc(sizeof(double) * S);
    orc_delta(M, S, T, delta);
    #pragma omp parallel for schedule(dynamic, 1)
    for (int h = 0; h < NH; ++h) {
        size_t ok = (size_t)h * L * dk, ov = (size_t)h * L * dv;
        head_backward(&c, delta, form == 3, q + ok, k + ok, v + ov, dout + ov, dq + ok, dk_ + ok, dv_ + ov);
    }
    free(delta);
    return 0;
}

int orc_max_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
