// decode.cu -- single-token BLA decode step (Alg. 2 loop body), bandwidth bound.
//
// One CTA of 256 threads (8 warps) per (batch, head).  The fp32 state is streamed
// twice, once for K and once for V, with 16-byte loads and stores that bypass L1
// (every state byte is read and written exactly once per step):
//   K pass: Z_m <- e^{i m w} Z_m + k (Eq. recurrence), y_m = q . Z_m
//   slots : s_j = scale sum_m c_m Re(e^{-i m w D_j} y_m) = scale q . K~[j]   (Eq. compressed),
//           masked unless pos >= D_j, p = softmax(s)                          (Eq. output)
//   V pass: Z_m <- e^{i m w} Z_m + v, o = sum_m u_m^c Re Z_m + u_m^s Im Z_m,
//           u_m = sum_j p_j (A[j,m], B[j,m])  (= sum_j p_j V~[j] with the sums exchanged)
// The sine row of mode 0 never changes (sin(0) = 0) and is neither read nor written.
// Absolute form (Alg. 1): the slots read q . Zabs_m = e^{-i m w pos} y_m through c_m e^{+i m w D_j}
// (the phi table with its sine half negated), and the output coefficient u_m is multiplied by
// e^{-i m w pos}; the state and its update are the same as in the lag form.
#include "common.cuh"

namespace bla {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

template <int VEC> struct VecT;
template <> struct VecT<4> { using T = float4; };
template <> struct VecT<2> { using T = float2; };
template <> struct VecT<1> { using T = float; };

template <int VEC> __device__ __forceinline__ void ldv(const float *p, float (&x)[VEC]) {
    if constexpr (VEC == 4) {
        float4 t = __ldcs(reinterpret_cast<const float4 *>(p));
        x[0] = t.x; x[1] = t.y; x[2] = t.z; x[3] = t.w;
    } else if constexpr (VEC == 2) {
        float2 t = __ldcs(reinterpret_cast<const float2 *>(p));
        x[0] = t.x; x[1] = t.y;
    } else {
        x[0] = __ldcs(p);
    }
}

template <int VEC> __device__ __forceinline__ void stv(float *p, const float (&x)[VEC]) {
    if constexpr (VEC == 4) {
        __stcs(reinterpret_cast<float4 *>(p), make_float4(x[0], x[1], x[2], x[3]));
    } else if constexpr (VEC == 2) {
        __stcs(reinterpret_cast<float2 *>(p), make_float2(x[0], x[1]));
    } else {
        __stcs(p, x[0]);
    }
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

// (cos, sin)(m w pos) in fp64, rounded to fp32.
__device__ __forceinline__ float2 pos_phase(int m, long long pos, double w) {
    double sn, cs;
    sincos((double)m * w * (double)pos, &sn, &cs);
    return make_float2((float)cs, (float)sn);
}

// Modes handled per warp per batch of independent loads.
constexpr int kUnroll = 4;

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) k_decode(OpDims d, long long pos, Tables tb, const T *__restrict__ q,
                                                     const T *__restrict__ k, const T *__restrict__ v,
                                                     float *__restrict__ state, T *__restrict__ o) {
    constexpr int VEC = D / 32;
    const int M = d.M, R2 = d.R2, S = d.S;
    const int bh = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const double w = tables_for_head(tb, bh % d.H, d.w);   // this head's tables and mode frequency
    extern __shared__ float sm[];
    float *y = sm;                 // [R2]: q . Z rows, later u
    float *ps = y + R2;            // [S]: scores, later probabilities
    float *opart = ps + S;         // [kWarps][D]

    float *ZK = state + (size_t)bh * 2 * R2 * D;
    float *ZV = ZK + (size_t)R2 * D;
    const int e0 = lane * VEC;

    float qv[VEC], kv[VEC], vv[VEC];
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
        qv[i] = load_elem<T>(q, (size_t)bh * D + e0 + i);
        kv[i] = load_elem<T>(k, (size_t)bh * D + e0 + i);
        vv[i] = load_elem<T>(v, (size_t)bh * D + e0 + i);
    }

    // ---- K pass
    for (int m0 = warp; m0 < M; m0 += kWarps * kUnroll) {
        float zc[kUnroll][VEC], zs[kUnroll][VEC];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            int m = m0 + u * kWarps;
            if (m < M) {
                ldv<VEC>(ZK + (size_t)(2 * m) * D + e0, zc[u]);
                if (m > 0) ldv<VEC>(ZK + (size_t)(2 * m + 1) * D + e0, zs[u]);
                else {
#pragma unroll
                    for (int i = 0; i < VEC; ++i) zs[u][i] = 0.f;
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            int m = m0 + u * kWarps;
            if (m < M) {
                float c = tb.rot1[2 * m], s = tb.rot1[2 * m + 1];
                float nc[VEC], ns[VEC], yc = 0.f, ys = 0.f;
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    nc[i] = fmaf(c, zc[u][i], fmaf(-s, zs[u][i], kv[i]));
                    ns[i] = fmaf(s, zc[u][i], c * zs[u][i]);
                    yc = fmaf(qv[i], nc[i], yc);
                    ys = fmaf(qv[i], ns[i], ys);
                }
                stv<VEC>(ZK + (size_t)(2 * m) * D + e0, nc);
                if (m > 0) stv<VEC>(ZK + (size_t)(2 * m + 1) * D + e0, ns);
                yc = warp_sum(yc);
                ys = warp_sum(ys);
                if (lane == 0) {
                    y[2 * m] = yc;
                    y[2 * m + 1] = (m > 0) ? ys : 0.f;
                }
            }
        }
    }
    __syncthreads();
    // absolute form: y_m <- e^{-i m w pos} y_m
    if (d.absolute) {
        for (int m = threadIdx.x; m < M; m += kThreads) {
            const float2 f = pos_phase(m, pos, w);
            const float yc = y[2 * m], ys = y[2 * m + 1];
            y[2 * m] = f.x * yc + f.y * ys;
            y[2 * m + 1] = f.x * ys - f.y * yc;
        }
        __syncthreads();
    }

    // ---- slot scores: warp per slot, lanes across the R2 state rows (coalesced table reads)
    for (int j = warp; j < S; j += kWarps) {
        const float *ph = tb.phi + (size_t)j * R2;
        float acc = 0.f;
        for (int r = lane; r < R2; r += 32) acc = fmaf(ph[r], y[r], acc);
        acc = warp_sum(acc);
        if (lane == 0) ps[j] = (pos >= (long long)tb.delta[j]) ? acc * d.scale : -INFINITY;
    }
    __syncthreads();
    // ---- softmax over the S slots (warp 0); slot 0 (D_0 = 0) is always visible
    if (warp == 0) {
        float mx = -INFINITY;
        for (int j = lane; j < S; j += 32) mx = fmaxf(mx, ps[j]);
        mx = warp_max(mx);
        float sum = 0.f;
        for (int j = lane; j < S; j += 32) {
            float e = (ps[j] == -INFINITY) ? 0.f : expf(ps[j] - mx);
            ps[j] = e;
            sum += e;
        }
        sum = warp_sum(sum);
        float inv = 1.f / sum;
        __syncwarp();
        for (int j = lane; j < S; j += 32) ps[j] *= inv;
    }
    __syncthreads();
    // ---- u_r = sum_j p_j phi[j][r]  (thread per state row, coalesced over r)
    for (int r = threadIdx.x; r < R2; r += kThreads) {
        float acc = 0.f;
        for (int j = 0; j < S; ++j) acc = fmaf(ps[j], tb.phi[(size_t)j * R2 + r], acc);
        y[r] = acc;
    }
    __syncthreads();
    // absolute form: the coefficient uc - i us is multiplied by e^{-i m w pos}
    if (d.absolute) {
        for (int m = threadIdx.x; m < M; m += kThreads) {
            const float2 f = pos_phase(m, pos, w);
            const float uc = y[2 * m], us = y[2 * m + 1];
            y[2 * m] = f.x * uc - f.y * us;
            y[2 * m + 1] = f.y * uc + f.x * us;
        }
        __syncthreads();
    }

    // ---- V pass
    float oacc[VEC];
#pragma unroll
    for (int i = 0; i < VEC; ++i) oacc[i] = 0.f;
    for (int m0 = warp; m0 < M; m0 += kWarps * kUnroll) {
        float zc[kUnroll][VEC], zs[kUnroll][VEC];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            int m = m0 + u * kWarps;
            if (m < M) {
                ldv<VEC>(ZV + (size_t)(2 * m) * D + e0, zc[u]);
                if (m > 0) ldv<VEC>(ZV + (size_t)(2 * m + 1) * D + e0, zs[u]);
                else {
#pragma unroll
                    for (int i = 0; i < VEC; ++i) zs[u][i] = 0.f;
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            int m = m0 + u * kWarps;
            if (m < M) {
                float c = tb.rot1[2 * m], s = tb.rot1[2 * m + 1];
                float uc = y[2 * m], us = y[2 * m + 1];
                float nc[VEC], ns[VEC];
#pragma unroll
                for (int i = 0; i < VEC; ++i) {
                    nc[i] = fmaf(c, zc[u][i], fmaf(-s, zs[u][i], vv[i]));
                    ns[i] = fmaf(s, zc[u][i], c * zs[u][i]);
                    oacc[i] = fmaf(uc, nc[i], fmaf(us, ns[i], oacc[i]));
                }
                stv<VEC>(ZV + (size_t)(2 * m) * D + e0, nc);
                if (m > 0) stv<VEC>(ZV + (size_t)(2 * m + 1) * D + e0, ns);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < VEC; ++i) opart[warp * D + e0 + i] = oacc[i];
    __syncthreads();
    for (int e = threadIdx.x; e < D; e += kThreads) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) acc += opart[w * D + e];
        store_elem<T>(o, (size_t)bh * D + e, acc);
    }
}

template <typename T, int D>
cudaError_t launch_decode_t(const OpDims &d, long long pos, const Tables &t, const void *q, const void *k,
                            const void *v, float *state, void *o, cudaStream_t st) {
    const int smem = decode_smem_bytes(d);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(k_decode<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
    }
    ProfScope ps(BLA_K_DECODE, st);
    k_decode<T, D><<<d.B * d.H, kThreads, smem, st>>>(d, pos, t, (const T *)q, (const T *)k, (const T *)v, state,
                                                     (T *)o);
    return cudaGetLastError();
}

}  // namespace

int decode_smem_bytes(const OpDims &d) {
    return (int)(sizeof(float) * ((size_t)d.R2 + d.S + (size_t)kWarps * d.dk));
}

cudaError_t launch_decode(const OpDims &d, long long pos, const Tables &t, const void *q, const void *k,
                          const void *v, float *state, void *o, cudaStream_t st) {
    const bool bf = d.dtype == BLA_BF16;
    switch (d.dk) {
    case 32: return bf ? launch_decode_t<__nv_bfloat16, 32>(d, pos, t, q, k, v, state, o, st)
                       : launch_decode_t<float, 32>(d, pos, t, q, k, v, state, o, st);
    case 64: return bf ? launch_decode_t<__nv_bfloat16, 64>(d, pos, t, q, k, v, state, o, st)
                       : launch_decode_t<float, 64>(d, pos, t, q, k, v, state, o, st);
    case 128: return bf ? launch_decode_t<__nv_bfloat16, 128>(d, pos, t, q, k, v, state, o, st)
                        : launch_decode_t<float, 128>(d, pos, t, q, k, v, state, o, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace bla
