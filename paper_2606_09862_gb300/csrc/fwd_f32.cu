// fwd_f32.cu -- fp32 chunked forward on CUDA cores (no tensor cores: the fp32 path's
// 1e-4 parity budget rules out single-pass TF32).
//
// One CTA per (batch, head) walks the sequence chunk by chunk.  Within a chunk of
// n <= C tokens starting at t0, with W the state carried into the chunk (the lag-frame
// state of Eq. (recurrence) advanced one step, W_m = e^{i m w} Z_m(t0-1), stored as
// interleaved rows 2m = real, 2m+1 = imaginary):
//   P[t,u]   = q_t . k_u                       (u <= t; intra-chunk scores)
//   X_m(t)   = sum_u P[t,u] e^{-i m w u} + q_t . W_m
//   Y_m(t)   = e^{i m w t} X_m(t)   = q_t . Z_m(t0+t)       (Eq. states)
//   s[t,j]   = scale sum_m c_m Re(e^{-i m w D_j} Y_m(t))   = scale q_t . K~[j]   (Eq. compressed)
//   p        = softmax_j(s) with slots t0+t < D_j masked     (Eq. output)
//   U_m(t)   = sum_j p[t,j] c_m e^{-i m w D_j};   A~_m(t) = U_m(t) e^{i m w t}
//   o_t      = sum_u G[t,u] v_u + sum_m Re(A~_m(t) WV_m),   G[t,u] = sum_m Re(A~_m(t) e^{-i m w u})
//   W_next   = e^{i m w C} (W + sum_u e^{-i m w u} k_u)
// This is Alg. 2's per-token read-out with the sums over slots, modes and past
// tokens exchanged; every term is an exact rearrangement of Eqs. (recurrence),
// (compressed) and (output).
//
// Absolute form (Alg. 1): slot j weights key u by D_M(u - D_j) instead of D_M(t - u - D_j).
// Its scores read q_t . Zabs_m(t) = e^{-i m w (t0+t)} Y_m(t) = e^{-i m w t0} X_m(t) through
// the coefficients c_m e^{+i m w D_j} (the phi table with its sine half negated), and its
// output coefficient is U'_m(t) e^{-i m w t0}.  So both per-row rotations e^{i m w t} become
// the chunk-constant e^{-i m w t0}; everything else is unchanged.
#include "common.cuh"

namespace bla {

namespace {

struct F32Smem {
    float *Q, *K, *V, *P, *X, *Sc, *Ph;
};

__global__ void __launch_bounds__(256) k_forward_f32(OpDims d, int C, Tables tb, const float *__restrict__ q,
                                                     const float *__restrict__ k, const float *__restrict__ v,
                                                     float *__restrict__ o, float *__restrict__ lse,
                                                     float *__restrict__ state) {
    extern __shared__ float smem[];
    const int dk = d.dk, dv = d.dv, M = d.M, R2 = d.R2, S = d.S, L = d.L;
    const int bh = blockIdx.x;
    const int tid = threadIdx.x, nt = blockDim.x;
    F32Smem sm;
    sm.Q = smem;
    sm.K = sm.Q + C * dk;
    sm.V = sm.K + C * dk;
    sm.P = sm.V + C * dv;
    sm.X = sm.P + C * C;
    sm.Sc = sm.X + C * R2;
    sm.Ph = sm.Sc + C * S;   // [M][2] absolute form: (cos, sin)(-m w t0) of the current chunk

    const float *qh = q + (size_t)bh * L * dk, *kh = k + (size_t)bh * L * dk, *vh = v + (size_t)bh * L * dv;
    float *oh = o + (size_t)bh * L * dv;
    float *lh = lse ? lse + (size_t)bh * L : nullptr;
    float *WK = state + (size_t)bh * R2 * (dk + dv);
    float *WV = WK + (size_t)R2 * dk;
    const float *erel = tb.erel, *phi = tb.phi;
    const int *delta = tb.delta;

    for (int i = tid; i < R2 * (dk + dv); i += nt) WK[i] = 0.f;
    __syncthreads();

    for (int t0 = 0; t0 < L; t0 += C) {
        const int n = min(C, L - t0);
        for (int i = tid; i < n * dk; i += nt) {
            sm.Q[i] = qh[(size_t)t0 * dk + i];
            sm.K[i] = kh[(size_t)t0 * dk + i];
        }
        for (int i = tid; i < n * dv; i += nt) sm.V[i] = vh[(size_t)t0 * dv + i];
        if (d.absolute) {
            for (int m = tid; m < M; m += nt) {
                double sn, cs;
                sincos((double)m * d.w * (double)t0, &sn, &cs);
                sm.Ph[2 * m] = (float)cs;
                sm.Ph[2 * m + 1] = (float)-sn;
            }
        }
        __syncthreads();
        // P = tril(Q K^T)
        for (int i = tid; i < n * n; i += nt) {
            int t = i / n, u = i % n;
            float acc = 0.f;
            if (u <= t)
                for (int e = 0; e < dk; ++e) acc = fmaf(sm.Q[t * dk + e], sm.K[u * dk + e], acc);
            sm.P[t * C + u] = acc;
        }
        __syncthreads();
        // X, then Y = e^{i m w t} X
        for (int i = tid; i < n * M; i += nt) {
            int t = i / M, m = i % M;
            float xc = 0.f, xs = 0.f;
            for (int u = 0; u <= t; ++u) {
                float pu = sm.P[t * C + u];
                xc = fmaf(pu, erel[(u * M + m) * 2], xc);
                xs = fmaf(-pu, erel[(u * M + m) * 2 + 1], xs);
            }
            const float *wc = WK + (size_t)(2 * m) * dk, *ws = wc + dk;
            for (int e = 0; e < dk; ++e) {
                xc = fmaf(sm.Q[t * dk + e], wc[e], xc);
                xs = fmaf(sm.Q[t * dk + e], ws[e], xs);
            }
            const float *ph = d.absolute ? sm.Ph + 2 * m : erel + (t * M + m) * 2;
            float c = ph[0], s = ph[1];
            sm.X[t * R2 + 2 * m] = c * xc - s * xs;
            sm.X[t * R2 + 2 * m + 1] = s * xc + c * xs;
        }
        __syncthreads();
        // slot scores with the mask t0 + t >= D_j
        for (int i = tid; i < n * S; i += nt) {
            int t = i / S, j = i % S;
            float acc = 0.f;
            for (int r = 0; r < R2; ++r) acc = fmaf(phi[j * R2 + r], sm.X[t * R2 + r], acc);
            sm.Sc[t * S + j] = (t0 + t >= delta[j]) ? acc * d.scale : -INFINITY;
        }
        __syncthreads();
        // softmax over slots, one thread per token (slot 0 has D_0 = 0, so a row is never empty)
        for (int t = tid; t < n; t += nt) {
            float mx = -INFINITY;
            for (int j = 0; j < S; ++j) mx = fmaxf(mx, sm.Sc[t * S + j]);
            float sum = 0.f;
            for (int j = 0; j < S; ++j) {
                float e = (sm.Sc[t * S + j] == -INFINITY) ? 0.f : expf(sm.Sc[t * S + j] - mx);
                sm.Sc[t * S + j] = e;
                sum += e;
            }
            float inv = 1.f / sum;
            for (int j = 0; j < S; ++j) sm.Sc[t * S + j] *= inv;
            if (lh) lh[t0 + t] = mx + logf(sum);
        }
        __syncthreads();
        // A~' (real form of A~ with the imaginary part negated), overwriting Y
        for (int i = tid; i < n * M; i += nt) {
            int t = i / M, m = i % M;
            float uc = 0.f, us = 0.f;
            for (int j = 0; j < S; ++j) {
                float pj = sm.Sc[t * S + j];
                uc = fmaf(pj, phi[j * R2 + 2 * m], uc);
                us = fmaf(pj, phi[j * R2 + 2 * m + 1], us);
            }
            const float *ph = d.absolute ? sm.Ph + 2 * m : erel + (t * M + m) * 2;
            float c = ph[0], s = ph[1];
            sm.X[t * R2 + 2 * m] = c * uc + s * us;
            sm.X[t * R2 + 2 * m + 1] = c * us - s * uc;
        }
        __syncthreads();
        // G = tril(A~' Ebar), Ebar[2m][u] = cos(m w u), Ebar[2m+1][u] = -sin(m w u)
        for (int i = tid; i < n * n; i += nt) {
            int t = i / n, u = i % n;
            float acc = 0.f;
            if (u <= t)
                for (int m = 0; m < M; ++m)
                    acc += sm.X[t * R2 + 2 * m] * erel[(u * M + m) * 2] -
                           sm.X[t * R2 + 2 * m + 1] * erel[(u * M + m) * 2 + 1];
            sm.P[t * C + u] = acc;
        }
        __syncthreads();
        // O = G V + A~' WV
        for (int i = tid; i < n * dv; i += nt) {
            int t = i / dv, e = i % dv;
            float acc = 0.f;
            for (int u = 0; u <= t; ++u) acc = fmaf(sm.P[t * C + u], sm.V[u * dv + e], acc);
            for (int r = 0; r < R2; ++r) acc = fmaf(sm.X[t * R2 + r], WV[(size_t)r * dv + e], acc);
            oh[(size_t)(t0 + t) * dv + e] = acc;
        }
        __syncthreads();
        // carried state: W <- e^{i m w n'} (W + sum_u e^{-i m w u} x_u), n' = C for a full chunk;
        // after the last chunk the lag-frame state Z(L-1) = e^{i m w (n-1)} (W + ...) is kept.
        const int adv = (t0 + n < L) ? n : n - 1;
        for (int i = tid; i < M * (dk + dv); i += nt) {
            int m = i / (dk + dv), e = i % (dk + dv);
            const bool isk = e < dk;
            const int ee = isk ? e : e - dk, dd = isk ? dk : dv;
            float *Wc = (isk ? WK : WV) + (size_t)(2 * m) * dd + ee, *Ws = Wc + dd;
            const float *X = isk ? sm.K : sm.V;
            float ac = *Wc, as = *Ws;
            for (int u = 0; u < n; ++u) {
                float x = X[u * dd + ee];
                ac = fmaf(erel[(u * M + m) * 2], x, ac);
                as = fmaf(-erel[(u * M + m) * 2 + 1], x, as);
            }
            float c = erel[(adv * M + m) * 2], s = erel[(adv * M + m) * 2 + 1];
            *Wc = c * ac - s * as;
            *Ws = s * ac + c * as;
        }
        __syncthreads();
    }
}

}  // namespace

int forward_f32_smem_bytes(const OpDims &d, int C) {
    size_t f = (size_t)C * d.dk * 2 + (size_t)C * d.dv + (size_t)C * C + (size_t)C * d.R2 + (size_t)C * d.S +
               (size_t)d.R2;
    return (int)(f * sizeof(float));
}

size_t forward_f32_scratch_bytes(const OpDims &d, int C) {
    (void)C;
    return align_up(sizeof(float) * (size_t)d.B * d.H * d.R2 * (d.dk + d.dv), 256);
}

cudaError_t launch_forward_f32(const OpDims &d, int C, const Tables &t, const float *q, const float *k,
                               const float *v, float *o, float *lse, float *state_out, float *scratch,
                               cudaStream_t st) {
    int smem = forward_f32_smem_bytes(d, C);
    cudaError_t e = cudaFuncSetAttribute(k_forward_f32, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    float *state = state_out ? state_out : scratch;
    ProfScope ps(BLA_K_FWD_F32, st);
    k_forward_f32<<<d.B * d.H, 256, smem, st>>>(d, C, t, q, k, v, o, lse, state);
    return cudaGetLastError();
}

}  // namespace bla
