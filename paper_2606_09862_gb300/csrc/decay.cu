// decay.cu -- Alg. 1 with the state decay of Sec. 3.3 (forward over a sequence and one decode step).
//
// The decayed form keeps Alg. 1's slot-space state: per head, S slots of d_k keys and d_v values.
// Token t (absolute index) updates every slot j with the translated Dirichlet weight
// D_j(t) = D_M(t - Delta_j) (Alg. 1's "interpolate", Eq. compressed_simplified), and the previous
// content is multiplied by (1 - D_j(t)) first (Sec. 3.3):
//     K~[j] <- (1 - D_j(t)) K~[j] + D_j(t) k_t,      V~[j] likewise.
// The read-out is Alg. 1's: p = softmax_j(scale q_t . K~[j]) over the slots with t >= Delta_j,
// o_t = sum_j p_j V~[j].
//
// Each slot column of the state is an independent first-order linear recurrence, so the forward
// runs as scans over time with the state in registers (the decay factors take both signs and
// reach zero, so the chunked form that divides by cumulative products is not used):
//   k_decay_table  D_M(x) for every x = t - Delta_j the call needs, in fp64 from the closed form
//                  of Eq. (dirichlet), (2M-1) D_M(x) = sin((M - 1/2) w x) / sin(w x / 2), after
//                  reducing w x to (-pi, pi]; and the grid Delta_j = round(j T / S).
//   k_decay_kscan  one warp per (head, slot): lanes hold d_k/32 state columns; for 32 tokens at a
//                  time the partial dot products q_t . K~[j] are reduced across the lanes by a
//                  transposing butterfly, so lane l ends with token t0 + l's score.
//   k_decay_lse    one thread per token: masked log-sum-exp over the slots.
//   k_decay_vscan  one CTA per (head, 32 value columns): thread (g, c) holds column c of the 8
//                  slots of group g; p, D and the value columns of 16 tokens are staged in shared
//                  memory and the groups' partial outputs are summed there.
//   k_decay_decode one CTA per head for a single token: K rows updated and scored, softmax,
//                  V rows updated and accumulated; every state row is read and written once.
#include <math.h>

#include "decay.cuh"

namespace bla {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kSlotsPerWarpGroup = 8;   // slots per thread in the V scan
constexpr int kVTile = 16;              // tokens per V-scan shared-memory tile
constexpr int kDecodeWarps = 8;
constexpr int kKBatch = 8;              // tokens whose q, k rows the K scan loads ahead

// D_M(x) at mode frequency w, Eq. (dirichlet) in its closed form.  w x is reduced to (-pi, pi]
// first, where the ratio is well conditioned; at the kernel's peak (|sin| below 1e-9) D = 1 to
// within M^2 (w x)^2 / 6 < 1e-11.
__device__ double dirichlet_closed(int M, double w, double x) {
    const double two_pi = 6.283185307179586476925286766559;
    double th = w * x;
    th -= two_pi * rint(th / two_pi);
    const double sh = sin(0.5 * th);
    if (fabs(sh) < 1e-9) return 1.0;
    return sin(((double)M - 0.5) * th) / ((2.0 * M - 1.0) * sh);
}

__device__ __forceinline__ int grid_delta(int j, double T, int S) { return (int)rint((double)j * T / (double)S); }

// per_slot == 0: Dx[i] = D_M(x0 + i), i < n.   per_slot != 0: Dx[j] = D_M(x0 - Delta_j), j < S.
// Both: delta[j] = round(j T / S) (round half to even, the default rounding mode).  With per-head
// periods (hp.n > 0) head h writes its own Dx[h][...] and delta[h][S] at (T_h, w_h); otherwise the
// single (T, w) is used.
__global__ void k_decay_table(int M, HeadPeriods hp, double T, double w, int S, long long x0, int n, int per_slot,
                              float *Dx, int *delta) {
    const int nh = hp.n > 0 ? hp.n : 1;
    const int per = (per_slot ? S : n) + S;
    const long long total = (long long)per * nh;
    for (long long ii = blockIdx.x * (long long)blockDim.x + threadIdx.x; ii < total;
         ii += (long long)gridDim.x * blockDim.x) {
        const int h = (int)(ii / per), i = (int)(ii % per);
        const double Th = hp.n > 0 ? hp.T[h] : T, wh = hp.n > 0 ? hp.w[h] : w;
        float *Dh = Dx + (size_t)h * (per_slot ? S : n);
        int *dh = delta + (size_t)h * S;
        if (per_slot) {
            if (i < S) Dh[i] = (float)dirichlet_closed(M, wh, (double)(x0 - grid_delta(i, Th, S)));
            else dh[i - S] = grid_delta(i - S, Th, S);
        } else {
            if (i < n) Dh[i] = (float)dirichlet_closed(M, wh, (double)(x0 + i));
            else dh[i - n] = grid_delta(i - n, Th, S);
        }
    }
}

// CPL consecutive elements of a row, as fp32.
template <typename T, int CPL> __device__ __forceinline__ void load_cols(const T *p, float *out);
template <> __device__ __forceinline__ void load_cols<float, 1>(const float *p, float *o) { o[0] = *p; }
template <> __device__ __forceinline__ void load_cols<float, 2>(const float *p, float *o) {
    const float2 a = *reinterpret_cast<const float2 *>(p);
    o[0] = a.x; o[1] = a.y;
}
template <> __device__ __forceinline__ void load_cols<float, 4>(const float *p, float *o) {
    const float4 a = *reinterpret_cast<const float4 *>(p);
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
}
template <> __device__ __forceinline__ void load_cols<__nv_bfloat16, 1>(const __nv_bfloat16 *p, float *o) {
    o[0] = __bfloat162float(*p);
}
template <> __device__ __forceinline__ void load_cols<__nv_bfloat16, 2>(const __nv_bfloat16 *p, float *o) {
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(p);
    o[0] = __low2float(a); o[1] = __high2float(a);
}
template <> __device__ __forceinline__ void load_cols<__nv_bfloat16, 4>(const __nv_bfloat16 *p, float *o) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&u.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&u.y);
    o[0] = __low2float(a); o[1] = __high2float(a); o[2] = __low2float(b); o[3] = __high2float(b);
}

template <int CPL> __device__ __forceinline__ void load_f32(const float *p, float *o) { load_cols<float, CPL>(p, o); }
template <int CPL> __device__ __forceinline__ void store_f32(float *p, const float *v) {
    if constexpr (CPL == 4) *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    else if constexpr (CPL == 2) *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
    else *p = v[0];
}

// K scan.  Block = 8 warps; block b covers head b / nsb and slots 8 (b % nsb) + warp.
// Writes sc[head][j][t] = scale q_t . K~_t[j] for t < L and the final K half of the state.
template <typename T, int CPL>
__global__ void __launch_bounds__(256) k_decay_kscan(const T *__restrict__ q, const T *__restrict__ k,
                                                     const float *__restrict__ Dx, const int *__restrict__ delta,
                                                     int S, int L, int d, int dmax, int nsb, float scale,
                                                     int H, int hs_dx, int hs_delta,
                                                     const float *state_in, float *state_out, float *__restrict__ sc) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long bh = blockIdx.x / nsb;
    const int j = (blockIdx.x % nsb) * 8 + warp;
    if (j >= S) return;                       // whole warps only; no block-level synchronisation below
    const int hd = (int)(bh % H);             // this head's D_M table and grid (strides 0 when shared)
    Dx += (size_t)hd * hs_dx;
    delta += (size_t)hd * hs_delta;
    const int off = dmax - delta[j];          // Dx index of token t is t + off
    const size_t row0 = (size_t)bh * L * d + lane * CPL;
    const size_t st = (size_t)bh * S * 2 * d + (size_t)j * d + lane * CPL;   // K half, slot j
    float K[CPL];
    if (state_in) load_f32<CPL>(state_in + st, K);
    else {
#pragma unroll
        for (int e = 0; e < CPL; ++e) K[e] = 0.f;
    }
    float *srow = sc + ((size_t)bh * S + j) * L;
    for (int t0 = 0; t0 < L; t0 += 32) {
        // D = 0 past the end of the sequence: those steps leave the state as it is.
        const float Dl = (t0 + lane < L) ? Dx[t0 + lane + off] : 0.f;
        float part[32];
#pragma unroll
        for (int u8 = 0; u8 < 32; u8 += kKBatch) {
            // The rows of kKBatch tokens are loaded before any is used (rows past the end repeat the
            // last one), so a warp has 2 kKBatch loads in flight instead of two.
            float kv[kKBatch][CPL], qv[kKBatch][CPL];
#pragma unroll
            for (int i = 0; i < kKBatch; ++i) {
                const size_t r = (size_t)min(t0 + u8 + i, L - 1) * d;
                load_cols<T, CPL>(k + row0 + r, kv[i]);
                load_cols<T, CPL>(q + row0 + r, qv[i]);
            }
#pragma unroll
            for (int i = 0; i < kKBatch; ++i) {
                const float D = __shfl_sync(kFull, Dl, u8 + i);
                const float keep = 1.f - D;
                float dot = 0.f;
#pragma unroll
                for (int e = 0; e < CPL; ++e) {
                    K[e] = fmaf(keep, K[e], D * kv[i][e]);
                    dot = fmaf(qv[i][e], K[e], dot);
                }
                part[u8 + i] = dot;
            }
        }
        // Transposing butterfly: after the stage of width o, a lane with bit o set holds the sums of
        // entries i + o in part[i]; after all five, lane l holds entry l summed over the 32 lanes.
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) {
            const bool up = (lane & o) != 0;
#pragma unroll
            for (int i = 0; i < o; ++i) {
                const float send = up ? part[i] : part[i + o];
                const float mine = up ? part[i + o] : part[i];
                part[i] = mine + __shfl_xor_sync(kFull, send, o);
            }
        }
        if (t0 + lane < L) srow[t0 + lane] = part[0] * scale;
    }
    if (state_out) store_f32<CPL>(state_out + st, K);
}

// lse[head][t] = log sum_{j : pos0 + t >= Delta_j} exp(sc[head][j][t]).
__global__ void k_decay_lse(const float *__restrict__ sc, const int *__restrict__ delta, int S, int L, long long pos0,
                            long long n, int H, int hs_delta, float *__restrict__ lse) {
    const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    if (i >= n) return;
    const long long bh = i / L;
    const int t = (int)(i % L);
    delta += (size_t)(bh % H) * hs_delta;
    const float *col = sc + (size_t)bh * S * L + t;
    float m = -INFINITY, sum = 0.f;
    for (int j = 0; j < S; ++j) {
        if (pos0 + t < delta[j]) continue;
        const float x = col[(size_t)j * L];
        if (x > m) {
            sum = sum * expf(m - x) + 1.f;
            m = x;
        } else {
            sum += expf(x - m);
        }
    }
    lse[i] = m + logf(sum);
}

// V scan.  Block = 32 * ng threads for head b / ncb and value columns 32 (b % ncb) + lane;
// thread (g, lane) holds slots 8 g .. 8 g + 7 of its column.
template <typename T>
__global__ void __launch_bounds__(1024) k_decay_vscan(const T *__restrict__ v, const float *__restrict__ Dx, const int *__restrict__ delta,
                              const float *__restrict__ sc, const float *__restrict__ lse, int S, int L, int dk, int dv,
                              int dmax, int ncb, int ng, long long pos0, int H, int hs_dx, int hs_delta,
                              const float *state_in, float *state_out, T *__restrict__ o) {
    constexpr int G = kSlotsPerWarpGroup, TT = kVTile;
    extern __shared__ float4 smem4[];
    const int spad = ng * G, sp = spad + 4;            // row stride: a multiple of 4 floats
    float *Dt = reinterpret_cast<float *>(smem4);      // [TT][sp]
    float *Pt = Dt + TT * sp;                          // [TT][sp]
    float *red = Pt + TT * sp;                         // [TT][ng][32]
    float *Vt = red + TT * ng * 32;                    // [TT][32]: the block's value columns
    int *dl = reinterpret_cast<int *>(Vt + TT * 32);   // [spad]
    const int g = threadIdx.x >> 5, lane = threadIdx.x & 31, nthr = blockDim.x;
    const long long bh = blockIdx.x / ncb;
    const int c = (blockIdx.x % ncb) * 32 + lane;
    Dx += (size_t)(bh % H) * hs_dx;           // this head's D_M table and grid (strides 0 when shared)
    delta += (size_t)(bh % H) * hs_delta;
    for (int i = threadIdx.x; i < spad; i += nthr) dl[i] = i < S ? delta[i] : 0;
    const size_t vst = (size_t)bh * S * (dk + dv) + (size_t)S * dk + c;   // V half, column c
    float V[G];
#pragma unroll
    for (int jj = 0; jj < G; ++jj) {
        const int j = g * G + jj;
        V[jj] = (state_in && j < S) ? state_in[vst + (size_t)j * dv] : 0.f;
    }
    __syncthreads();
    const T *vb = v + (size_t)bh * L * dv + (c - lane);   // first column of the block
    T *oh = o + (size_t)bh * L * dv + c;
    const float *sh = sc + (size_t)bh * S * L;
    const float *lh = lse + (size_t)bh * L;
    for (int t0 = 0; t0 < L; t0 += TT) {
        for (int idx = threadIdx.x; idx < TT * spad; idx += nthr) {
            const int tt = idx % TT, j = idx / TT, t = t0 + tt;
            float D = 0.f, P = 0.f;
            if (j < S && t < L) {
                D = Dx[t + dmax - dl[j]];
                if (pos0 + t >= dl[j]) P = expf(sh[(size_t)j * L + t] - lh[t]);
            }
            Dt[tt * sp + j] = D;
            Pt[tt * sp + j] = P;
        }
        for (int idx = threadIdx.x; idx < TT * 32; idx += nthr) {
            const int t = t0 + (idx >> 5);
            Vt[idx] = t < L ? load_elem<T>(vb, (size_t)t * dv + (idx & 31)) : 0.f;
        }
        __syncthreads();
        const int nt = min(TT, L - t0);
#pragma unroll 4
        for (int tt = 0; tt < nt; ++tt) {
            const float x = Vt[tt * 32 + lane];
            const float4 *d4 = reinterpret_cast<const float4 *>(Dt + tt * sp + g * G);
            const float4 *p4 = reinterpret_cast<const float4 *>(Pt + tt * sp + g * G);
            const float4 da = d4[0], db = d4[1], pa = p4[0], pb = p4[1];
            const float dd[G] = {da.x, da.y, da.z, da.w, db.x, db.y, db.z, db.w};
            const float pp[G] = {pa.x, pa.y, pa.z, pa.w, pb.x, pb.y, pb.z, pb.w};
            float acc = 0.f;
#pragma unroll
            for (int jj = 0; jj < G; ++jj) {
                V[jj] = fmaf(1.f - dd[jj], V[jj], dd[jj] * x);
                acc = fmaf(pp[jj], V[jj], acc);
            }
            red[(tt * ng + g) * 32 + lane] = acc;
        }
        __syncthreads();
        for (int tt = g; tt < nt; tt += ng) {
            float s = 0.f;
            for (int gg = 0; gg < ng; ++gg) s += red[(tt * ng + gg) * 32 + lane];
            store_elem<T>(oh, (size_t)(t0 + tt) * dv, s);
        }
    }
    if (state_out) {
#pragma unroll
        for (int jj = 0; jj < G; ++jj) {
            const int j = g * G + jj;
            if (j < S) state_out[vst + (size_t)j * dv] = V[jj];
        }
    }
}

// One decode step.  Block = 8 warps, one head; warp w takes slots w, w + 8, ... two at a time so
// that two state rows are in flight per warp.
template <typename T, int CPL>
__global__ void __launch_bounds__(256) k_decay_decode(const T *__restrict__ q, const T *__restrict__ k,
                                                      const T *__restrict__ v, const float *__restrict__ Dj,
                                                      const int *__restrict__ delta, int S, int d, long long pos,
                                                      float scale, int H, int hs, float *__restrict__ state,
                                                      T *__restrict__ o) {
    __shared__ float s_sc[256];
    __shared__ float s_red[kDecodeWarps][128];
    __shared__ float s_stat[2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long bh = blockIdx.x;
    Dj += (size_t)(bh % H) * hs;              // this head's weights D_j(pos) and grid (stride 0 when shared)
    delta += (size_t)(bh % H) * hs;
    float *Ks = state + (size_t)bh * 2 * S * d + lane * CPL;
    float *Vs = Ks + (size_t)S * d;
    float qv[CPL], kv[CPL], vv[CPL];
    load_cols<T, CPL>(q + (size_t)bh * d + lane * CPL, qv);
    load_cols<T, CPL>(k + (size_t)bh * d + lane * CPL, kv);
    load_cols<T, CPL>(v + (size_t)bh * d + lane * CPL, vv);
    for (int j0 = warp; j0 < S; j0 += 2 * kDecodeWarps) {
        const int j1 = j0 + kDecodeWarps;
        const bool two = j1 < S;
        float a[CPL], b[CPL] = {};
        load_f32<CPL>(Ks + (size_t)j0 * d, a);
        if (two) load_f32<CPL>(Ks + (size_t)j1 * d, b);
        const float D0 = Dj[j0], D1 = two ? Dj[j1] : 0.f;
        float s0 = 0.f, s1 = 0.f;
#pragma unroll
        for (int e = 0; e < CPL; ++e) {
            a[e] = fmaf(1.f - D0, a[e], D0 * kv[e]);
            s0 = fmaf(qv[e], a[e], s0);
            b[e] = fmaf(1.f - D1, b[e], D1 * kv[e]);
            s1 = fmaf(qv[e], b[e], s1);
        }
        store_f32<CPL>(Ks + (size_t)j0 * d, a);
        if (two) store_f32<CPL>(Ks + (size_t)j1 * d, b);
#pragma unroll
        for (int o2 = 16; o2 >= 1; o2 >>= 1) {
            s0 += __shfl_xor_sync(kFull, s0, o2);
            s1 += __shfl_xor_sync(kFull, s1, o2);
        }
        if (lane == 0) {
            s_sc[j0] = pos >= delta[j0] ? s0 * scale : -INFINITY;
            if (two) s_sc[j1] = pos >= delta[j1] ? s1 * scale : -INFINITY;
        }
    }
    __syncthreads();
    if (warp == 0) {
        float m = -INFINITY;
        for (int j = lane; j < S; j += 32) m = fmaxf(m, s_sc[j]);
#pragma unroll
        for (int o2 = 16; o2 >= 1; o2 >>= 1) m = fmaxf(m, __shfl_xor_sync(kFull, m, o2));
        float sum = 0.f;
        for (int j = lane; j < S; j += 32) sum += expf(s_sc[j] - m);   // masked slots: exp(-inf) = 0
#pragma unroll
        for (int o2 = 16; o2 >= 1; o2 >>= 1) sum += __shfl_xor_sync(kFull, sum, o2);
        if (lane == 0) {
            s_stat[0] = m;
            s_stat[1] = 1.f / sum;
        }
    }
    __syncthreads();
    const float m = s_stat[0], inv = s_stat[1];
    float acc[CPL];
#pragma unroll
    for (int e = 0; e < CPL; ++e) acc[e] = 0.f;
    for (int j0 = warp; j0 < S; j0 += 2 * kDecodeWarps) {
        const int j1 = j0 + kDecodeWarps;
        const bool two = j1 < S;
        float a[CPL], b[CPL] = {};
        load_f32<CPL>(Vs + (size_t)j0 * d, a);
        if (two) load_f32<CPL>(Vs + (size_t)j1 * d, b);
        const float D0 = Dj[j0], D1 = two ? Dj[j1] : 0.f;
        const float p0 = expf(s_sc[j0] - m) * inv, p1 = two ? expf(s_sc[j1] - m) * inv : 0.f;
#pragma unroll
        for (int e = 0; e < CPL; ++e) {
            a[e] = fmaf(1.f - D0, a[e], D0 * vv[e]);
            b[e] = fmaf(1.f - D1, b[e], D1 * vv[e]);
            acc[e] = fmaf(p0, a[e], acc[e]);
            acc[e] = fmaf(p1, b[e], acc[e]);
        }
        store_f32<CPL>(Vs + (size_t)j0 * d, a);
        if (two) store_f32<CPL>(Vs + (size_t)j1 * d, b);
    }
#pragma unroll
    for (int e = 0; e < CPL; ++e) s_red[warp][lane * CPL + e] = acc[e];
    __syncthreads();
    for (int col = threadIdx.x; col < d; col += blockDim.x) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < kDecodeWarps; ++w) s += s_red[w][col];
        store_elem<T>(o, (size_t)bh * d + col, s);
    }
}

// ------------------------------------------------------------------ backward (VJP)
// Unrolled, the decayed slot state is a fixed linear map of the tokens,
//     K~_j(t) = sum_{u<=t} W_j(t,u) k_u,     W_j(t,u) = D_j(u) prod_{u<x<=t} (1 - D_j(x)),
// so the chain rule through s = scale q . K~, the masked softmax and o = sum_j p V~ gives, with
// upstream do:
//     dp[t,j] = do_t . V~_j(t),     g[t,j] = scale p[t,j] (dp[t,j] - do_t . o_t)
//     dq_t = sum_j g[t,j] K~_j(t)                                                  forward in time
//     lK_j(t) = g[t,j] q_t + (1 - D_j(t+1)) lK_j(t+1),    dk_t = sum_j D_j(t) lK_j(t)    backward
//     lV_j(t) = p[t,j] do_t + (1 - D_j(t+1)) lV_j(t+1),   dv_t = sum_j D_j(t) lV_j(t)    backward
// dp comes from the K scan with (do, v) in place of (q, k); the three sums over slots run in
// k_decay_rscan, the V scan's layout with the per-token factors (f, u, w) of
//     X_j <- f X_j + u x_t,     out_t = sum_j w X_j
// staged per tile: forward in time f = 1 - D_j(t), u = D_j(t), w = g; backward in time
// f = 1 - D_j(t+1), u = g or p, w = D_j(t).

// g[head][j][t] = scale p (dp - do_t . o_t), in place of dp; one thread per token.
template <typename T>
__global__ void k_decay_ds(const float *__restrict__ sc, const float *__restrict__ lse, float *__restrict__ g,
                           const T *__restrict__ dout, const T *__restrict__ o, const int *__restrict__ delta, int S,
                           int L, int dv, long long pos0, float scale, long long n, int H, int hs_delta) {
    const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    if (i >= n) return;
    const long long bh = i / L;
    const int t = (int)(i % L);
    delta += (size_t)(bh % H) * hs_delta;
    float rd = 0.f;
    for (int c = 0; c < dv; ++c) rd = fmaf(load_elem<T>(dout, (size_t)i * dv + c), load_elem<T>(o, (size_t)i * dv + c), rd);
    const size_t col = (size_t)bh * S * L + t;
    const float l = lse[i];
    for (int j = 0; j < S; ++j) {
        const size_t e = col + (size_t)j * L;
        g[e] = (pos0 + t >= delta[j]) ? scale * expf(sc[e] - l) * (g[e] - rd) : 0.f;
    }
}

// Reduce scan over the slots for 32 columns of one head (layout of k_decay_vscan).  REV = false:
// forward in time, f = 1 - D_j(t), u = D_j(t), w = wt(t, j).  REV = true: backward in time,
// f = 1 - D_j(t+1), u = wt(t, j), w = D_j(t).  wt(t, j) = G[j][t] when lse is NULL, else the slot
// probability exp(G[j][t] - lse[t]) (G holding scores; 0 on masked slots).
template <typename T, bool REV>
__global__ void __launch_bounds__(1024) k_decay_rscan(const T *__restrict__ x, const float *__restrict__ Dx,
                                                      const int *__restrict__ delta, const float *__restrict__ G,
                                                      const float *__restrict__ lse, int S, int L, int dx, int dmax,
                                                      int ncb, int ng, long long pos0, int H, int hs_dx, int hs_delta,
                                                      T *__restrict__ out) {
    constexpr int G8 = kSlotsPerWarpGroup, TT = kVTile;
    extern __shared__ float4 smem4[];
    const int spad = ng * G8, sp = spad + 4;
    float *Ft = reinterpret_cast<float *>(smem4);      // [TT][sp]
    float *Ut = Ft + TT * sp;                          // [TT][sp]
    float *Wt = Ut + TT * sp;                          // [TT][sp]
    float *red = Wt + TT * sp;                         // [TT][ng][32]
    float *Xt = red + TT * ng * 32;                    // [TT][32]
    int *dl = reinterpret_cast<int *>(Xt + TT * 32);   // [spad]
    const int g = threadIdx.x >> 5, lane = threadIdx.x & 31, nthr = blockDim.x;
    const long long bh = blockIdx.x / ncb;
    const int c = (blockIdx.x % ncb) * 32 + lane;
    Dx += (size_t)(bh % H) * hs_dx;           // this head's D_M table and grid (strides 0 when shared)
    delta += (size_t)(bh % H) * hs_delta;
    for (int i = threadIdx.x; i < spad; i += nthr) dl[i] = i < S ? delta[i] : 0;
    float X[G8];
#pragma unroll
    for (int jj = 0; jj < G8; ++jj) X[jj] = 0.f;
    __syncthreads();
    const T *xb = x + (size_t)bh * L * dx + (c - lane);
    T *oh = out + (size_t)bh * L * dx + c;
    const float *gh = G + (size_t)bh * S * L;
    const float *lh = lse ? lse + (size_t)bh * L : nullptr;
    for (int t0 = 0; t0 < L; t0 += TT) {
        // tile position tt holds token t = t0 + tt (forward) or L - 1 - (t0 + tt) (backward)
        for (int idx = threadIdx.x; idx < TT * spad; idx += nthr) {
            const int tt = idx % TT, j = idx / TT, r = t0 + tt;
            float f = 0.f, u = 0.f, w = 0.f;
            if (j < S && r < L) {
                const int t = REV ? L - 1 - r : r;
                float wt;
                if (lh) wt = (pos0 + t >= dl[j]) ? expf(gh[(size_t)j * L + t] - lh[t]) : 0.f;
                else wt = gh[(size_t)j * L + t];
                const float Dt = Dx[t + dmax - dl[j]];
                if (REV) {
                    f = 1.f - Dx[t + 1 + dmax - dl[j]];   // entry L + dmax - Delta_j < L + dmax + 1 at t = L - 1
                    u = wt;
                    w = Dt;
                } else {
                    f = 1.f - Dt;
                    u = Dt;
                    w = wt;
                }
            }
            Ft[tt * sp + j] = f;
            Ut[tt * sp + j] = u;
            Wt[tt * sp + j] = w;
        }
        for (int idx = threadIdx.x; idx < TT * 32; idx += nthr) {
            const int r = t0 + (idx >> 5);
            const int t = REV ? L - 1 - r : r;
            Xt[idx] = r < L ? load_elem<T>(xb, (size_t)t * dx + (idx & 31)) : 0.f;
        }
        __syncthreads();
        const int nt = min(TT, L - t0);
#pragma unroll 4
        for (int tt = 0; tt < nt; ++tt) {
            const float xv = Xt[tt * 32 + lane];
            const float4 *f4 = reinterpret_cast<const float4 *>(Ft + tt * sp + g * G8);
            const float4 *u4 = reinterpret_cast<const float4 *>(Ut + tt * sp + g * G8);
            const float4 *w4 = reinterpret_cast<const float4 *>(Wt + tt * sp + g * G8);
            const float4 fa = f4[0], fb = f4[1], ua = u4[0], ub = u4[1], wa = w4[0], wb = w4[1];
            const float ff[G8] = {fa.x, fa.y, fa.z, fa.w, fb.x, fb.y, fb.z, fb.w};
            const float uu[G8] = {ua.x, ua.y, ua.z, ua.w, ub.x, ub.y, ub.z, ub.w};
            const float ww[G8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
            float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
            for (int jj = 0; jj < G8; jj += 2) {
                X[jj] = fmaf(ff[jj], X[jj], uu[jj] * xv);
                X[jj + 1] = fmaf(ff[jj + 1], X[jj + 1], uu[jj + 1] * xv);
                acc0 = fmaf(ww[jj], X[jj], acc0);
                acc1 = fmaf(ww[jj + 1], X[jj + 1], acc1);
            }
            red[(tt * ng + g) * 32 + lane] = acc0 + acc1;
        }
        __syncthreads();
        for (int tt = g; tt < nt; tt += ng) {
            float sum = 0.f;
            for (int gg = 0; gg < ng; ++gg) sum += red[(tt * ng + gg) * 32 + lane];
            const int r = t0 + tt;
            store_elem<T>(oh, (size_t)(REV ? L - 1 - r : r) * dx, sum);
        }
    }
}

// Largest Delta_j (the grid is non-decreasing in j), computed exactly as the device does.
int host_dmax(const OpDims &d) { return (int)rint((double)(d.S - 1) * d.T / (double)d.S); }

struct DecayWs {
    int *delta;      // [nh][S]
    float *Dx;       // [nh][S] (decode) or [nh][L + max Delta + 1] (forward)
    float *sc;
    float *lse;
    int hs_dx, hs_delta;   // per-head strides of Dx and delta (0 when the heads share one period)
    float *g = nullptr;    // backward: dp, then g = scale ds, [BH][S][L]
    // chunked forward and backward (decay_chunk.cu): chunk states, adjoint contributions and tables
    void *chunk = nullptr;
};

size_t decay_table_len(const OpDims &d) { return (size_t)d.L + (size_t)host_dmax(d) + 1; }

size_t carve(const OpDims &d, bool decode, bool own_lse, char *base, DecayWs *w, bool backward = false) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += align_up(bytes, 256);
        return p;
    };
    const size_t nh = d.periods ? (size_t)d.H : 1;
    const size_t per = decode ? (size_t)d.S : decay_table_len(d);
    w->delta = reinterpret_cast<int *>(take(sizeof(int) * nh * d.S));
    w->Dx = reinterpret_cast<float *>(take(sizeof(float) * nh * per));
    w->hs_dx = d.periods ? (int)per : 0;
    w->hs_delta = d.periods ? d.S : 0;
    w->sc = nullptr;
    w->lse = nullptr;
    if (!decode && backward && decay_chunk_supported(d)) {
        w->chunk = take(decay_chunk_bwd_ws_bytes(d));
    } else if (!decode && !backward && decay_chunk_supported(d)) {
        // the chunked forward keeps its scores on chip: the chunk states and tables travel
        if (own_lse) w->lse = reinterpret_cast<float *>(take(sizeof(float) * (size_t)d.B * d.H * (size_t)d.L));
        w->chunk = take(decay_chunk_fwd_ws_bytes(d));
    } else if (!decode) {
        const size_t BH = (size_t)d.B * d.H;
        w->sc = reinterpret_cast<float *>(take(sizeof(float) * BH * d.S * (size_t)(d.L > 0 ? d.L : 1)));
        if (own_lse) w->lse = reinterpret_cast<float *>(take(sizeof(float) * BH * (size_t)(d.L > 0 ? d.L : 1)));
        w->g = backward ? reinterpret_cast<float *>(take(sizeof(float) * BH * d.S * (size_t)(d.L > 0 ? d.L : 1)))
                        : nullptr;
    }
    return off;
}

template <typename T>
cudaError_t kscan_dispatch(const OpDims &d, const DecayWs &w, const void *q, const void *k, int dmax,
                           const float *state_in, float *state_out, cudaStream_t st) {
    const int nsb = (d.S + 7) / 8;
    const long long blocks = (long long)d.B * d.H * nsb;
    const T *qq = static_cast<const T *>(q), *kk = static_cast<const T *>(k);
    ProfScope ps(BLA_K_DECAY, st);
    switch (d.dk) {
    case 32: k_decay_kscan<T, 1><<<(unsigned)blocks, 256, 0, st>>>(qq, kk, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    d.scale, d.H, w.hs_dx, w.hs_delta, state_in,
                                                                    state_out, w.sc); break;
    case 64: k_decay_kscan<T, 2><<<(unsigned)blocks, 256, 0, st>>>(qq, kk, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    d.scale, d.H, w.hs_dx, w.hs_delta, state_in,
                                                                    state_out, w.sc); break;
    default: k_decay_kscan<T, 4><<<(unsigned)blocks, 256, 0, st>>>(qq, kk, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    d.scale, d.H, w.hs_dx, w.hs_delta, state_in,
                                                                    state_out, w.sc); break;
    }
    return cudaGetLastError();
}

size_t vscan_smem(int ng) {
    const int spad = ng * kSlotsPerWarpGroup, sp = spad + 4;
    return sizeof(float) * ((size_t)2 * kVTile * sp + (size_t)kVTile * ng * 32 + (size_t)kVTile * 32) +
           sizeof(int) * (size_t)spad;
}

template <typename T>
cudaError_t vscan_dispatch(const OpDims &d, const DecayWs &w, const float *lse, const void *v, void *o, int dmax,
                           long long pos0, const float *state_in, float *state_out, cudaStream_t st) {
    const int ncb = d.dv / 32;
    const int ng = (d.S + kSlotsPerWarpGroup - 1) / kSlotsPerWarpGroup;
    const size_t smem = vscan_smem(ng);
    cudaError_t e = cudaFuncSetAttribute(k_decay_vscan<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long blocks = (long long)d.B * d.H * ncb;
    ProfScope ps(BLA_K_DECAY, st);
    k_decay_vscan<T><<<(unsigned)blocks, 32 * ng, smem, st>>>(static_cast<const T *>(v), w.Dx, w.delta, w.sc, lse,
                                                              d.S, d.L, d.dk, d.dv, dmax, ncb, ng, pos0, d.H, w.hs_dx,
                                                              w.hs_delta, state_in, state_out, static_cast<T *>(o));
    return cudaGetLastError();
}

cudaError_t table_launch(const OpDims &d, long long x0, int n, int per_slot, const DecayWs &w, cudaStream_t st) {
    HeadPeriods hp;
    head_periods(d, d.omega_in, &hp);   // hp.n = 0 when the heads share one period
    const long long total = (long long)((per_slot ? d.S : n) + d.S) * (hp.n > 0 ? hp.n : 1);
    long long blocks = (total + 255) / 256;
    if (blocks > 1024) blocks = 1024;
    ProfScope ps(BLA_K_DECAY, st);
    k_decay_table<<<(int)blocks, 256, 0, st>>>(d.M, hp, d.T, d.w, d.S, x0, n, per_slot, w.Dx, w.delta);
    return cudaGetLastError();
}

// K scan with explicit operands: out[head][j][t] = scale z_t . X_j(t), X_j <- (1 - D) X_j + D x_t.
template <typename T>
cudaError_t kscan_launch(const OpDims &d, const DecayWs &w, const void *z, const void *x, int dmax, float scale,
                         float *out, cudaStream_t st) {
    const int nsb = (d.S + 7) / 8;
    const long long blocks = (long long)d.B * d.H * nsb;
    const T *zz = static_cast<const T *>(z), *xx = static_cast<const T *>(x);
    ProfScope ps(BLA_K_DECAY, st);
    switch (d.dk) {
    case 32: k_decay_kscan<T, 1><<<(unsigned)blocks, 256, 0, st>>>(zz, xx, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    scale, d.H, w.hs_dx, w.hs_delta, nullptr, nullptr,
                                                                    out); break;
    case 64: k_decay_kscan<T, 2><<<(unsigned)blocks, 256, 0, st>>>(zz, xx, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    scale, d.H, w.hs_dx, w.hs_delta, nullptr, nullptr,
                                                                    out); break;
    default: k_decay_kscan<T, 4><<<(unsigned)blocks, 256, 0, st>>>(zz, xx, w.Dx, w.delta, d.S, d.L, d.dk, dmax, nsb,
                                                                    scale, d.H, w.hs_dx, w.hs_delta, nullptr, nullptr,
                                                                    out); break;
    }
    return cudaGetLastError();
}

size_t rscan_smem(int ng) {
    const int spad = ng * kSlotsPerWarpGroup, sp = spad + 4;
    return sizeof(float) * ((size_t)3 * kVTile * sp + (size_t)kVTile * ng * 32 + (size_t)kVTile * 32) +
           sizeof(int) * (size_t)spad;
}

template <typename T, bool REV>
cudaError_t rscan_launch(const OpDims &d, const DecayWs &w, const void *x, const float *G, const float *lse, int dmax,
                         long long pos0, void *out, cudaStream_t st) {
    const int ncb = d.dv / 32;
    const int ng = (d.S + kSlotsPerWarpGroup - 1) / kSlotsPerWarpGroup;
    const size_t smem = rscan_smem(ng);
    cudaError_t e = cudaFuncSetAttribute(k_decay_rscan<T, REV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long blocks = (long long)d.B * d.H * ncb;
    ProfScope ps(BLA_K_DECAY, st);
    k_decay_rscan<T, REV><<<(unsigned)blocks, 32 * ng, smem, st>>>(static_cast<const T *>(x), w.Dx, w.delta, G, lse,
                                                                   d.S, d.L, d.dv, dmax, ncb, ng, pos0, d.H, w.hs_dx,
                                                                   w.hs_delta, static_cast<T *>(out));
    return cudaGetLastError();
}

template <typename T>
cudaError_t backward_run(const OpDims &d, const DecayWs &w, long long pos0, const void *q, const void *k,
                         const void *v, const void *o, const void *dout, const float *lse, void *dq, void *dk,
                         void *dv, int dmax, cudaStream_t st) {
    cudaError_t e;
    if ((e = kscan_launch<T>(d, w, q, k, dmax, d.scale, w.sc, st)) != cudaSuccess) return e;    // scores
    if ((e = kscan_launch<T>(d, w, dout, v, dmax, 1.f, w.g, st)) != cudaSuccess) return e;     // dp
    const long long nt = (long long)d.B * d.H * d.L;
    {
        ProfScope ps(BLA_K_DECAY, st);
        k_decay_ds<T><<<(unsigned)((nt + 255) / 256), 256, 0, st>>>(w.sc, lse, w.g, static_cast<const T *>(dout),
                                                                    static_cast<const T *>(o), w.delta, d.S, d.L,
                                                                    d.dv, pos0, d.scale, nt, d.H, w.hs_delta);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if ((e = rscan_launch<T, false>(d, w, k, w.g, nullptr, dmax, pos0, dq, st)) != cudaSuccess) return e;
    if ((e = rscan_launch<T, true>(d, w, q, w.g, nullptr, dmax, pos0, dk, st)) != cudaSuccess) return e;
    return rscan_launch<T, true>(d, w, dout, w.sc, lse, dmax, pos0, dv, st);
}

}  // namespace

size_t decay_backward_workspace_bytes(const OpDims &d) {
    DecayWs w;
    return carve(d, false, false, nullptr, &w, true);
}

cudaError_t launch_decay_backward(const OpDims &d, long long pos0, const void *q, const void *k, const void *v,
                                  const void *o, const void *dout, const float *lse, void *dq, void *dk, void *dv,
                                  void *ws, cudaStream_t st) {
    if (d.L == 0) return cudaSuccess;
    DecayWs w;
    carve(d, false, false, static_cast<char *>(ws), &w, true);
    const int dmax = host_dmax(d);
    cudaError_t e = table_launch(d, pos0 - dmax, (int)decay_table_len(d), 0, w, st);
    if (e != cudaSuccess) return e;
    if (decay_chunk_supported(d))
        return launch_decay_chunk_bwd(d, pos0, dmax, w.Dx, w.delta, w.hs_dx, w.hs_delta, q, k, v, dout, lse, dq, dk,
                                      dv, w.chunk, st);
    return d.dtype == BLA_BF16 ? backward_run<__nv_bfloat16>(d, w, pos0, q, k, v, o, dout, lse, dq, dk, dv, dmax, st)
                               : backward_run<float>(d, w, pos0, q, k, v, o, dout, lse, dq, dk, dv, dmax, st);
}

size_t decay_table_entries(const OpDims &d) { return decay_table_len(d); }

size_t decay_workspace_bytes(const OpDims &d, bool decode) {
    DecayWs w;
    return carve(d, decode, true, nullptr, &w);
}

cudaError_t launch_decay_forward(const OpDims &d, long long pos0, const void *q, const void *k, const void *v, void *o,
                                 float *lse, const float *state_in, float *state_out, void *ws, cudaStream_t st) {
    DecayWs w;
    carve(d, false, lse == nullptr, static_cast<char *>(ws), &w);
    const int dmax = host_dmax(d);
    const int n = (int)decay_table_len(d);
    cudaError_t e = table_launch(d, pos0 - dmax, n, 0, w, st);
    if (e != cudaSuccess) return e;
    if (decay_chunk_supported(d))
        return launch_decay_chunk(d, pos0, dmax, w.Dx, w.delta, w.hs_dx, w.hs_delta, q, k, v, o, lse ? lse : w.lse,
                                  state_in, state_out, w.chunk, st);
    e = d.dtype == BLA_BF16 ? kscan_dispatch<__nv_bfloat16>(d, w, q, k, dmax, state_in, state_out, st)
                            : kscan_dispatch<float>(d, w, q, k, dmax, state_in, state_out, st);
    if (e != cudaSuccess) return e;
    float *l = lse ? lse : w.lse;
    const long long nt = (long long)d.B * d.H * d.L;
    if (nt > 0) {
        ProfScope ps(BLA_K_DECAY, st);
        k_decay_lse<<<(unsigned)((nt + 255) / 256), 256, 0, st>>>(w.sc, w.delta, d.S, d.L, pos0, nt, d.H, w.hs_delta, l);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return d.dtype == BLA_BF16 ? vscan_dispatch<__nv_bfloat16>(d, w, l, v, o, dmax, pos0, state_in, state_out, st)
                               : vscan_dispatch<float>(d, w, l, v, o, dmax, pos0, state_in, state_out, st);
}

cudaError_t launch_decay_decode(const OpDims &d, long long pos, const void *q, const void *k, const void *v,
                                float *state, void *o, void *ws, cudaStream_t st) {
    DecayWs w;
    carve(d, true, false, static_cast<char *>(ws), &w);
    cudaError_t e = table_launch(d, pos, 0, 1, w, st);
    if (e != cudaSuccess) return e;
    const unsigned blocks = (unsigned)((long long)d.B * d.H);
    ProfScope ps(BLA_K_DECAY, st);
    if (d.dtype == BLA_BF16) {
        using T = __nv_bfloat16;
        const T *qq = static_cast<const T *>(q), *kk = static_cast<const T *>(k), *vv = static_cast<const T *>(v);
        T *oo = static_cast<T *>(o);
        switch (d.dk) {
        case 32: k_decay_decode<T, 1><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        case 64: k_decay_decode<T, 2><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        default: k_decay_decode<T, 4><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        }
    } else {
        using T = float;
        const T *qq = static_cast<const T *>(q), *kk = static_cast<const T *>(k), *vv = static_cast<const T *>(v);
        T *oo = static_cast<T *>(o);
        switch (d.dk) {
        case 32: k_decay_decode<T, 1><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        case 64: k_decay_decode<T, 2><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        default: k_decay_decode<T, 4><<<blocks, 256, 0, st>>>(qq, kk, vv, w.Dx, w.delta, d.S, d.dk, pos, d.scale, d.H, w.hs_delta, state, oo); break;
        }
    }
    return cudaGetLastError();
}

}  // namespace bla
