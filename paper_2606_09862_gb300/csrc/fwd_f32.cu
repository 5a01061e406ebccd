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

// stage != 0: the phase and slot tables (also transposed, for the loops that walk them across
// rows) and the carried state live in shared memory, copied in at the start, the state written out
// at the end; otherwise they are read from global memory.  Rows of the q, k, v tiles (and of the
// staged state) are padded by one float so that loops over rows do not hit one bank.
__global__ void __launch_bounds__(256) k_forward_f32(OpDims d, int C, Tables tb, const float *__restrict__ q,
                                                     const float *__restrict__ k, const float *__restrict__ v,
                                                     float *__restrict__ o, float *__restrict__ lse,
                                                     float *__restrict__ state, int stage) {
    extern __shared__ float smem[];
    const int dk = d.dk, dv = d.dv, M = d.M, R2 = d.R2, S = d.S, L = d.L;
    const int QS = dk + 1, VS = dv + 1;   // padded row strides of the q/k and v tiles
    const int bh = blockIdx.x;
    const int tid = threadIdx.x, nt = blockDim.x;
    const double w = tables_for_head(tb, bh % d.H, d.w);   // this head's tables and mode frequency
    F32Smem sm;
    sm.Q = smem;
    sm.K = sm.Q + C * QS;
    sm.V = sm.K + C * QS;
    sm.P = sm.V + C * VS;
    sm.X = sm.P + C * C;
    sm.Sc = sm.X + C * R2;
    sm.Ph = sm.Sc + C * S;   // [M][2] absolute form: (cos, sin)(-m w t0) of the current chunk
    float *st_erel = sm.Ph + R2, *st_erelT = st_erel + (C + 1) * M * 2, *st_phi = st_erelT + (C + 1) * M * 2;
    float *st_phiT = st_phi + S * R2, *st_state = st_phiT + S * R2;

    const float *qh = q + (size_t)bh * L * dk, *kh = k + (size_t)bh * L * dk, *vh = v + (size_t)bh * L * dv;
    float *oh = o + (size_t)bh * L * dv;
    float *lh = lse ? lse + (size_t)bh * L : nullptr;
    float *const gstate = state + (size_t)bh * R2 * (dk + dv);
    // carried state: rows of the K part, then the V part, row strides KS / VSt
    const int KS = stage ? dk + 1 : dk, VSt = stage ? dv + 1 : dv;
    float *WK = stage ? st_state : gstate;
    float *WV = WK + (size_t)R2 * KS;
    // phase table erel[(u M + m) 2 + c] and slot table phi[j R2 + r]; eT(u, m) and phT(r, j) index
    // their transposes when staged (the plain tables otherwise)
    const float *erel = tb.erel, *phi = tb.phi, *erelT = tb.erel, *phiT = tb.phi;
    const int *delta = tb.delta;
    if (stage) {
        for (int i = tid; i < (C + 1) * M; i += nt) {
            const int u = i / M, m = i % M;
            const float c = tb.erel[2 * i], s = tb.erel[2 * i + 1];
            st_erel[2 * i] = c;
            st_erel[2 * i + 1] = s;
            st_erelT[(m * (C + 1) + u) * 2] = c;
            st_erelT[(m * (C + 1) + u) * 2 + 1] = s;
        }
        for (int i = tid; i < S * R2; i += nt) {
            const float x = tb.phi[i];
            st_phi[i] = x;
            st_phiT[(i % R2) * S + i / R2] = x;
        }
        erel = st_erel;
        phi = st_phi;
        erelT = st_erelT;
        phiT = st_phiT;
    }
    auto eT = [&](int u, int m, int comp) {
        return stage ? erelT[(m * (C + 1) + u) * 2 + comp] : erel[(u * M + m) * 2 + comp];
    };
    auto phT = [&](int r, int j) { return stage ? phiT[r * S + j] : phi[j * R2 + r]; };

    for (int i = tid; i < R2 * KS + R2 * VSt; i += nt) WK[i] = 0.f;
    __syncthreads();

    for (int t0 = 0; t0 < L; t0 += C) {
        const int n = min(C, L - t0);
        for (int i = tid; i < n * dk; i += nt) {
            const int r = i / dk, c = i % dk;
            sm.Q[r * QS + c] = qh[(size_t)t0 * dk + i];
            sm.K[r * QS + c] = kh[(size_t)t0 * dk + i];
        }
        for (int i = tid; i < n * dv; i += nt) sm.V[(i / dv) * VS + i % dv] = vh[(size_t)t0 * dv + i];
        if (d.absolute) {
            for (int m = tid; m < M; m += nt) {
                double sn, cs;
                sincos((double)m * w * (double)t0, &sn, &cs);
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
                for (int e = 0; e < dk; ++e) acc = fmaf(sm.Q[t * QS + e], sm.K[u * QS + e], acc);
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
            const float *wc = WK + (size_t)(2 * m) * KS, *ws = wc + KS;
            for (int e = 0; e < dk; ++e) {
                xc = fmaf(sm.Q[t * QS + e], wc[e], xc);
                xs = fmaf(sm.Q[t * QS + e], ws[e], xs);
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
            for (int r = 0; r < R2; ++r) acc = fmaf(phT(r, j), sm.X[t * R2 + r], acc);
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
                    acc += sm.X[t * R2 + 2 * m] * eT(u, m, 0) - sm.X[t * R2 + 2 * m + 1] * eT(u, m, 1);
            sm.P[t * C + u] = acc;
        }
        __syncthreads();
        // O = G V + A~' WV
        for (int i = tid; i < n * dv; i += nt) {
            int t = i / dv, e = i % dv;
            float acc = 0.f;
            for (int u = 0; u <= t; ++u) acc = fmaf(sm.P[t * C + u], sm.V[u * VS + e], acc);
            for (int r = 0; r < R2; ++r) acc = fmaf(sm.X[t * R2 + r], WV[(size_t)r * VSt + e], acc);
            oh[(size_t)(t0 + t) * dv + e] = acc;
        }
        __syncthreads();
        // carried state: W <- e^{i m w n'} (W + sum_u e^{-i m w u} x_u), n' = C for a full chunk;
        // after the last chunk the lag-frame state Z(L-1) = e^{i m w (n-1)} (W + ...) is kept.
        const int adv = (t0 + n < L) ? n : n - 1;
        for (int i = tid; i < M * (dk + dv); i += nt) {
            int m = i / (dk + dv), e = i % (dk + dv);
            const bool isk = e < dk;
            const int ee = isk ? e : e - dk, xs_ = isk ? QS : VS, ws_ = isk ? KS : VSt;
            float *Wc = (isk ? WK : WV) + (size_t)(2 * m) * ws_ + ee, *Ws = Wc + ws_;
            const float *X = isk ? sm.K : sm.V;
            float ac = *Wc, as = *Ws;
            for (int u = 0; u < n; ++u) {
                float x = X[u * xs_ + ee];
                ac = fmaf(erel[(u * M + m) * 2], x, ac);
                as = fmaf(-erel[(u * M + m) * 2 + 1], x, as);
            }
            float c = erel[(adv * M + m) * 2], s = erel[(adv * M + m) * 2 + 1];
            *Wc = c * ac - s * as;
            *Ws = s * ac + c * as;
        }
        __syncthreads();
    }
    if (stage) {
        // out to the global layout [R2][dk] then [R2][dv]
        for (int i = tid; i < R2 * dk; i += nt) gstate[i] = WK[(i / dk) * KS + i % dk];
        for (int i = tid; i < R2 * dv; i += nt) gstate[R2 * dk + i] = WV[(i / dv) * VSt + i % dv];
    }
}

}  // namespace

int forward_f32_smem_bytes(const OpDims &d, int C) {
    size_t f = (size_t)C * (d.dk + 1) * 2 + (size_t)C * (d.dv + 1) + (size_t)C * C + (size_t)C * d.R2 +
               (size_t)C * d.S + (size_t)d.R2;
    return (int)(f * sizeof(float));
}

// Extra shared memory of the staged variant: the phase table and the slot table (each also
// transposed), and the carried state with padded rows.
static int forward_f32_stage_bytes(const OpDims &d, int C) {
    size_t f = 2 * (size_t)(C + 1) * d.M * 2 + 2 * (size_t)d.S * d.R2 + (size_t)d.R2 * (d.dk + 1 + d.dv + 1);
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
    const int staged = smem + forward_f32_stage_bytes(d, C);
    const int stage = staged <= 227 * 1024;
    if (stage) smem = staged;
    cudaError_t e = cudaFuncSetAttribute(k_forward_f32, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    float *state = state_out ? state_out : scratch;
    ProfScope ps(BLA_K_FWD_F32, st);
    k_forward_f32<<<d.B * d.H, 256, smem, st>>>(d, C, t, q, k, v, o, lse, state, stage);
    return cudaGetLastError();
}

}  // namespace bla
