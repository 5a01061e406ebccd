// bwd.cu -- backward pass of the chunked forward (vector-Jacobian product for q, k, v).
//
// The forward of a chunk (see fwd_bf16.cu) is, with W_K, W_V the states entering it,
//   P = tril(Q K^T), Y = rot+(P EB^T + Q W_K^T), p = softmax(scale Y PHI^T),
//   A' = rot-(p PHI), G = tril(A' EB), O = G V + A' W_V,   W_next = rot_C(W + EB X).
// Its adjoint, given dO, is
//   dG = tril(dO V^T), dU = rot+(dG EB^T + dO W_V^T), dp = dU PHI^T, ds = p (dp - rowsum(dO o)),
//   dX = rot-(scale ds PHI), dP = tril(dX EB),
//   dQ = dP K + dX W_K,  dK = dP^T Q + EB^T Lk,  dV = G^T dO + EB^T Lv,
// where the adjoint states L of the chunk sums (W + EB X) run backwards over the chunks:
//   L_{c-1} = rot_C^T (X_c^T + L_c) with X_c^T = dX^T Q (K) or A'^T dO (V), L_last = 0.
//
// Every contraction runs on the tensor cores through one batched kernel, k_bgemm: one CTA per
// (chunk, 128-row tile) computes sum_t A_t B_t (up to two terms) with A, B streamed by TMA in
// 64-wide K blocks through a shared-memory ring, accumulates in TMEM and applies a fused
// epilogue (causal mask, per-mode phase rotation, probability recompute from lse, dS, addend).
// The forward chunk states and the adjoint states come from element-wise scans on CUDA cores.
//
// Absolute form (Alg. 1): the forward's two per-row rotations by m w tau become one rotation by
// -m w t0 (t0 = the chunk's first token) and PHI has its sine half negated (see fwd_f32.cu).  The
// adjoint rotations are the transposes at the same angle, so every EP_ROT epilogue takes its
// phase from a per-chunk table instead of the per-row one; the rest of the backward is shared.
#include <math.h>
#include <string.h>

#include "bwd.cuh"
#include "fwd_bf16.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace bla {

namespace {

using bf16 = __nv_bfloat16;
constexpr int kC = 128;
constexpr int kThreads = 192;

enum OpMode { OP_SHARED = 0, OP_Z = 1, OP_SEQ = 2 };
enum EpiOp { EP_PLAIN = 0, EP_CAUSAL, EP_ROT, EP_PROB, EP_DS, EP_ADD };
enum OutMode { OUT_Z = 0, OUT_SEQ = 1 };

struct Operand {
    int mode;     // OpMode
    int kmajor;   // 1: rows = M (A) or N (B), K contiguous;  0: K rows, M/N contiguous
    int zmul, zoff;
    int mn_off;   // offset on the M/N axis (A also gets + 128 * M-tile)
};

struct Term {
    Operand A, B;
    int K;        // multiple of 64
};

struct Epi {
    int op, rot_sign;
    float scale;
    int out_mode, out_f32, ldo, ncols_out;
    int out_rows;            // rows per output block (OUT_Z); rows at or beyond it are skipped
    int out_zmul, out_zoff;  // output block index = z * out_zmul + out_zoff
    void *out;
    const float *lse;        // EP_PROB: [BH][L]
    const int *delta;        // EP_PROB: [S]
    int S;
    const bf16 *pbuf;        // EP_DS: [Z][128][ldp]
    int ldp;
    const float *dl;         // EP_DS: [Z][128]
    const float *addend;     // EP_ADD: [Z][128][ldo] fp32
    const float *erel;       // EP_ROT: (cos, sin)(m w tau), [C+1][M][2]
    const float *cphase;     // EP_ROT, absolute form: (cos, sin)(-m w c C), [nchunks][M][2] (else null)
    int M;
};

struct GemmArgs {
    int nterms;
    Term t[2];
    int N;
    int BH, L, nchunks;
    Epi e;
    int *err;
};

struct Ctl {
    volatile int abort;
};

__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t &phase, Ctl *ctl, int *err, int which) {
    if (ctl->abort) return false;
    bool ok = tc::mbar_wait(bar, phase);
    if (!ok) {
        ctl->abort = 1;
        report_device_error(err, DEVERR_MBAR_TIMEOUT | (4 << 4) | (which << 8) | ((int)phase << 15) |
                                     ((int)blockIdx.x << 16));
    }
    phase ^= 1u;
    return ok;
}

__device__ __forceinline__ uint64_t kmaj_desc(uint32_t base, int k) {
    return tc::sdesc_sw128(base + (uint32_t)(k * 32), 16, 1024);
}
__device__ __forceinline__ uint64_t mnmaj_desc(uint32_t base, int k) {
    return tc::sdesc_sw128(base + (uint32_t)(k * 16 * 128), 64u * 128u, 1024);
}

// TMA loads of one 64-wide K block of an operand with M/N extent R into `dst`.
__device__ __forceinline__ void load_block(const CUtensorMap *map, const Operand &op, int R, int kb, int mn_extra,
                                           int z, int bh, int c, uint8_t *dst, uint64_t *bar) {
    const int mn0 = op.mn_off + mn_extra;
    if (op.kmajor) {
        if (op.mode == OP_SHARED) tc::tma_load_2d(dst, map, bar, kb * 64, mn0);
        else if (op.mode == OP_Z) tc::tma_load_3d(dst, map, bar, kb * 64, mn0, z * op.zmul + op.zoff);
        else tc::tma_load_3d(dst, map, bar, kb * 64, c * kC + mn0, bh);
    } else {
        for (int nb = 0; nb < R / 64; ++nb) {
            uint8_t *d = dst + nb * 64 * 128;
            if (op.mode == OP_SHARED) tc::tma_load_2d(d, map, bar, mn0 + nb * 64, kb * 64);
            else if (op.mode == OP_Z) tc::tma_load_3d(d, map, bar, mn0 + nb * 64, kb * 64, z * op.zmul + op.zoff);
            else tc::tma_load_3d(d, map, bar, mn0 + nb * 64, c * kC + kb * 64, bh);
        }
    }
}

constexpr int kMaxStages = 4;

// Persistent: CTA i takes tiles i, i + gridDim.x, ... (tile = (z, 128-row M tile), z fastest
// within an M tile).  The producer streams every tile's K blocks through one shared-memory ring;
// the MMA issuer alternates between two TMEM accumulators, so the epilogue drains tile j while
// the MMAs of tile j+1 run.
__global__ void __launch_bounds__(kThreads, 1)
    k_bgemm(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mB0,
            const __grid_constant__ CUtensorMap mA1, const __grid_constant__ CUtensorMap mB1, GemmArgs g, int stages,
            int ntiles) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int N = g.N;
    const size_t a_bytes = (size_t)kC * 64 * 2, b_bytes = (size_t)N * 64 * 2;
    const size_t stage_bytes = a_bytes + b_bytes;
    uint64_t *full = reinterpret_cast<uint64_t *>(sm + stages * stage_bytes);
    uint64_t *empty = full + kMaxStages;
    uint64_t *acc_full = empty + kMaxStages;   // [2]
    uint64_t *acc_empty = acc_full + 2;        // [2], one arrival per epilogue warp
    uint32_t *tslot = reinterpret_cast<uint32_t *>(acc_empty + 2);
    Ctl *ctl = reinterpret_cast<Ctl *>(acc_empty + 3);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t ncols = N <= 16 ? 32u : N <= 32 ? 64u : N <= 64 ? 128u : N <= 128 ? 256u : 512u;   // 2 x N
    const int kb0 = g.t[0].K / 64, nkb = kb0 + (g.nterms > 1 ? g.t[1].K / 64 : 0);
    const int Z = g.BH * g.nchunks;

    if (threadIdx.x == 0) {
        for (int i = 0; i < stages; ++i) { tc::mbar_init(&full[i], 1); tc::mbar_init(&empty[i], 1); }
        for (int i = 0; i < 2; ++i) { tc::mbar_init(&acc_full[i], 1); tc::mbar_init(&acc_empty[i], 4); }
        ctl->abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 5) { tc::tmem_alloc(tslot, ncols); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;

    if (warp == 4 && lane == 0) {
        uint32_t ph[kMaxStages] = {0, 0, 0, 0};
        long long it = 0;   // K blocks issued so far, over all tiles of this CTA
        bool bad = false;
        for (int tile = blockIdx.x; tile < ntiles && !bad; tile += gridDim.x) {
            const int z = tile % Z, mt = tile / Z;
            const int bh = z / g.nchunks, c = z % g.nchunks;
            for (int kk = 0; kk < nkb; ++kk, ++it) {
                const int st = (int)(it % stages);
                if (it >= stages && !wait_bar(&empty[st], ph[st], ctl, g.err, 1)) { bad = true; break; }
                const int term = kk < kb0 ? 0 : 1, kb = kk < kb0 ? kk : kk - kb0;
                const Term &t = g.t[term];
                uint8_t *base = sm + st * stage_bytes;
                tc::mbar_arrive_expect_tx(&full[st], (uint32_t)stage_bytes);
                load_block(term ? &mA1 : &mA0, t.A, kC, kb, mt * kC, z, bh, c, base, &full[st]);
                load_block(term ? &mB1 : &mB0, t.B, N, kb, 0, z, bh, c, base + a_bytes, &full[st]);
            }
        }
    } else if (warp == 5 && lane == 0) {
        uint32_t ph[kMaxStages] = {0, 0, 0, 0}, ph_ae[2] = {0, 0};
        long long it = 0;
        int j = 0;   // tiles of this CTA so far
        bool bad = false;
        for (int tile = blockIdx.x; tile < ntiles && !bad; tile += gridDim.x, ++j) {
            const int buf = j & 1;
            // the accumulator's previous tile (j - 2) must have been drained
            if (j >= 2 && !wait_bar(&acc_empty[buf], ph_ae[buf], ctl, g.err, 4)) break;
            const uint32_t acc = tb + (uint32_t)(buf * N);
            for (int kk = 0; kk < nkb; ++kk, ++it) {
                const int st = (int)(it % stages);
                if (!wait_bar(&full[st], ph[st], ctl, g.err, 2)) { bad = true; break; }
                tc::tc_fence_after();
                const int term = kk < kb0 ? 0 : 1;
                const Term &t = g.t[term];
                const uint32_t idesc = tc::idesc_bf16(128, N, !t.A.kmajor, !t.B.kmajor);
                const uint32_t a = tc::smem_u32(sm + st * stage_bytes), b = a + (uint32_t)a_bytes;
                for (int k = 0; k < 4; ++k)
                    tc::mma_bf16(acc, t.A.kmajor ? kmaj_desc(a, k) : mnmaj_desc(a, k),
                                 t.B.kmajor ? kmaj_desc(b, k) : mnmaj_desc(b, k), idesc, (kk > 0 || k > 0) ? 1u : 0u);
                tc::mma_commit(&empty[st]);
            }
            tc::mma_commit(&acc_full[buf]);
        }
    } else if (warp < 4) {
        uint32_t ph_af[2] = {0, 0};
        int j = 0;
        for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++j) {
            const int buf = j & 1;
            const int z = tile % Z, mt = tile / Z;
            const int bh = z / g.nchunks, c = z % g.nchunks;
            if (!wait_bar(&acc_full[buf], ph_af[buf], ctl, g.err, 3)) break;
            tc::tc_fence_after();
            const uint32_t tacc = tb + (uint32_t)(buf * N);
            {
            const Epi &e = g.e;
            const int row = threadIdx.x, lane_base = warp * 32;
            const int orow = mt * kC + row;
            const int t = c * kC + row;                  // token index (rows are chunk tokens)
            const bool live = (e.out_mode == OUT_SEQ) ? (t < g.L) : (orow < e.out_rows);
            char *obase = nullptr;
            if (e.out_mode == OUT_Z)
                obase = (char *)e.out + (((size_t)(z * e.out_zmul + e.out_zoff) * e.out_rows + orow) * e.ldo) *
                                            (e.out_f32 ? 4 : 2);
            else
                obase = (char *)e.out + (((size_t)bh * g.L + t) * e.ldo) * (e.out_f32 ? 4 : 2);
            const float lse = (e.op == EP_PROB && t < g.L) ? e.lse[(size_t)bh * g.L + t] : 0.f;
            const float dl = (e.op == EP_DS) ? e.dl[(size_t)z * kC + row] : 0.f;
            for (int g0 = 0; g0 < e.ncols_out; g0 += 32) {
                float v[32];
                if (g0 < N) tc::tmem_ld32(tacc + ((uint32_t)lane_base << 16) + (uint32_t)g0, v);
                else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = 0.f;
                }
                if (g0 < N) {
                    if (e.op == EP_CAUSAL) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (g0 + i > row) v[i] = 0.f;
                    } else if (e.op == EP_ROT) {
                        // e^{i m w row} for the 16 modes of this block: the table's first phase, then
                        // products with e^{i w row} (16 steps; rounding far below bf16 resolution)
                        // (absolute form: e^{-i m w t0} of the chunk, stepped by e^{-i w t0})
                        const int m0 = g0 >> 1;
                        const float *ptab = e.cphase ? e.cphase + (size_t)c * e.M * 2 : e.erel + (size_t)row * e.M * 2;
                        float cs = ptab[m0 * 2], sn = ptab[m0 * 2 + 1];
                        const float c1 = ptab[2], s1 = ptab[3];
#pragma unroll
                        for (int i = 0; i < 32; i += 2) {
                            const float sg = e.rot_sign * sn;
                            const float xr = v[i], xi = v[i + 1];
                            v[i] = e.scale * (cs * xr - sg * xi);
                            v[i + 1] = e.scale * (sg * xr + cs * xi);
                            const float t = cs * c1 - sn * s1;
                            sn = sn * c1 + cs * s1;
                            cs = t;
                        }
                    } else if (e.op == EP_PROB) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int j = g0 + i;
                            v[i] = (t < g.L && j < e.S && t >= e.delta[j]) ? __expf(e.scale * v[i] - lse) : 0.f;
                        }
                    } else if (e.op == EP_DS) {
                        const bf16 *pr = e.pbuf + ((size_t)z * kC + row) * e.ldp + g0;
#pragma unroll
                        for (int i = 0; i < 32; i += 8) {
                            const uint4 pk = __ldg(reinterpret_cast<const uint4 *>(pr + i));
                            const uint32_t w[4] = {pk.x, pk.y, pk.z, pk.w};
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const float2 pf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[q]));
                                v[i + 2 * q] = pf.x * (v[i + 2 * q] - dl);
                                v[i + 2 * q + 1] = pf.y * (v[i + 2 * q + 1] - dl);
                            }
                        }
                    } else if (e.op == EP_ADD) {
                        const float *ad = e.addend + ((size_t)z * kC + row) * e.ldo + g0;
#pragma unroll
                        for (int i = 0; i < 32; i += 4) {
                            const float4 a4 = __ldg(reinterpret_cast<const float4 *>(ad + i));
                            v[i] += a4.x;
                            v[i + 1] += a4.y;
                            v[i + 2] += a4.z;
                            v[i + 3] += a4.w;
                        }
                    }
                }
                if (!live) continue;
                if (e.out_f32) {
                    float *o = reinterpret_cast<float *>(obase) + g0;
#pragma unroll
                    for (int i = 0; i < 32; i += 4) *reinterpret_cast<float4 *>(o + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                } else {
                    bf16 *o = reinterpret_cast<bf16 *>(obase) + g0;
#pragma unroll
                    for (int i = 0; i < 32; i += 8)
                        *reinterpret_cast<uint4 *>(o + i) =
                            make_uint4(tc::pack_bf16x2(v[i], v[i + 1]), tc::pack_bf16x2(v[i + 2], v[i + 3]),
                                       tc::pack_bf16x2(v[i + 4], v[i + 5]), tc::pack_bf16x2(v[i + 6], v[i + 7]));
                }
            }
            }
            // the accumulator may take tile j + 2
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&acc_empty[buf]);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 5) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, ncols);
    }
}

// ------------------------------------------------------------------ scans (CUDA cores)

// Forward chunk states: W_0 = 0, W_{c+1} = rot_C (W_c + contrib_c); writes bf16 W_c for every chunk.
// contrib, wout: [Z][2][R2][D] with Z = BH * nchunks.  One thread per (bh, x, m, e).
__global__ void k_state_scan(int BH, int nch, int M, int D, const float *erel, const float *contrib, bf16 *wout,
                             int reverse) {
    const long long total = (long long)BH * 2 * M * D;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int e = (int)(i % D);
        long long r = i / D;
        const int m = (int)(r % M);
        r /= M;
        const int x = (int)(r % 2);
        const int bh = (int)(r / 2);
        const int R2 = 2 * M;
        const float cs = erel[((size_t)kC * M + m) * 2], sn = erel[((size_t)kC * M + m) * 2 + 1];
        float re = 0.f, im = 0.f;
        // the contributions of eight chunks are loaded before they are used, so that their
        // latencies overlap
        for (int s0 = 0; s0 < nch; s0 += 8) {
            float cr[8], ci[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                cr[j] = ci[j] = 0.f;
                if (s0 + j < nch) {
                    const int c = reverse ? nch - 1 - (s0 + j) : s0 + j;
                    const size_t base = (((size_t)bh * nch + c) * 2 + x) * R2;
                    cr[j] = __ldg(contrib + (base + 2 * m) * D + e);
                    ci[j] = __ldg(contrib + (base + 2 * m + 1) * D + e);
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (s0 + j >= nch) break;
                const int c = reverse ? nch - 1 - (s0 + j) : s0 + j;
                const size_t base = (((size_t)bh * nch + c) * 2 + x) * R2;
                wout[(base + 2 * m) * D + e] = __float2bfloat16_rn(re);
                wout[(base + 2 * m + 1) * D + e] = __float2bfloat16_rn(im);
                const float ar = re + cr[j], ai = im + ci[j];
                if (!reverse) {          // rot by +m w C
                    re = cs * ar - sn * ai;
                    im = sn * ar + cs * ai;
                } else {                 // transpose: rot by -m w C
                    re = cs * ar + sn * ai;
                    im = -sn * ar + cs * ai;
                }
            }
        }
    }
}
// Absolute form: (cos, sin)(-m w c C) for every chunk c and mode m, in fp64 rounded to fp32.
__global__ void k_chunk_phase(int M, int nch, double w, float *out) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nch * M; i += gridDim.x * blockDim.x) {
        const int c = i / M, m = i % M;
        double sn, cs;
        sincos((double)m * w * ((double)c * kC), &sn, &cs);
        out[2 * i] = (float)cs;
        out[2 * i + 1] = (float)-sn;
    }
}

// rowsum(dO o) per token: one warp per row, each lane reading D/32 consecutive elements.
__global__ void k_rowdot(int BH, int L, int nch, int D, const bf16 *dout, const bf16 *o, float *dl) {
    const long long rows = (long long)BH * nch * kC;
    const int lane = threadIdx.x & 31;
    const long long warps = (long long)gridDim.x * (blockDim.x >> 5);
    for (long long i = blockIdx.x * (long long)(blockDim.x >> 5) + (threadIdx.x >> 5); i < rows; i += warps) {
        const int row = (int)(i % kC);
        const long long z = i / kC;
        const int bh = (int)(z / nch), c = (int)(z % nch);
        const int t = c * kC + row;
        float acc = 0.f;
        if (t < L) {
            const bf16 *a = dout + ((size_t)bh * L + t) * D, *b = o + ((size_t)bh * L + t) * D;
            for (int j = lane * 2; j < D; j += 64) {
                const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(a + j));
                const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(b + j));
                acc = fmaf(x.x, y.x, fmaf(x.y, y.y, acc));
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
        if (lane == 0) dl[i] = acc;
    }
}

// ------------------------------------------------------------------ host side

struct BwdGeo {
    int BH, L, D, M, R2, RP, S, SP, nch, Z;
};

BwdGeo bwd_geo(const OpDims &d) {
    BwdGeo g;
    g.BH = d.B * d.H; g.L = d.L; g.D = d.dk; g.M = d.M; g.R2 = d.R2;
    g.RP = d.R2 <= 128 ? 128 : d.R2;
    g.S = d.S; g.SP = d.S < 64 ? 64 : d.S;
    g.nch = (d.L + kC - 1) / kC;
    g.Z = g.BH * g.nch;
    return g;
}

struct BwdWs {
    size_t tables, eb, phi, cphase, cb, wb, lb, P, Y, p, A, G, dG, dU, ds, dX, dP, dKi, dVi, dl, total;
};

BwdWs bwd_ws(const OpDims &d, const BwdGeo &g) {
    BwdWs w;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off += align_up(bytes, 1024); return o; };
    const size_t Z = (size_t)g.Z;
    w.tables = take(tables_bytes(d, kC));
    w.eb = take(2 * (size_t)g.RP * kC);
    w.phi = take(2 * (size_t)g.SP * g.R2);
    w.cphase = take(d.absolute ? 4 * (size_t)g.nch * g.M * 2 : 0);
    w.cb = take(4 * Z * 2 * g.R2 * g.D);
    w.wb = take(2 * Z * 2 * g.R2 * g.D);
    w.lb = take(2 * Z * 2 * g.R2 * g.D);
    w.P = take(2 * Z * kC * kC);
    w.Y = take(2 * Z * kC * g.R2);
    w.p = take(2 * Z * kC * g.SP);
    w.A = take(2 * Z * kC * g.R2);
    w.G = take(2 * Z * kC * kC);
    w.dG = take(2 * Z * kC * kC);
    w.dU = take(2 * Z * kC * g.R2);
    w.ds = take(2 * Z * kC * g.SP);
    w.dX = take(2 * Z * kC * g.R2);
    w.dP = take(2 * Z * kC * kC);
    w.dKi = take(4 * Z * kC * g.D);
    w.dVi = take(4 * Z * kC * g.D);
    w.dl = take(4 * Z * kC);
    w.total = off;
    return w;
}

// Tensor maps: K-major operand of R rows -> box {64, R}; MN-major -> box {64, 64}.
bool map_seq(CUtensorMap *m, const void *p, const BwdGeo &g, int cols, bool kmajor, int R) {
    const uint64_t dims[3] = {(uint64_t)cols, (uint64_t)g.L, (uint64_t)g.BH};
    const uint64_t str[2] = {(uint64_t)cols * 2, (uint64_t)g.L * cols * 2};
    const uint32_t box[3] = {64, (uint32_t)(kmajor ? R : 64), 1};
    return make_tmap_bf16(m, p, 3, dims, str, box);
}
bool map_z(CUtensorMap *m, const void *p, int cols, int rows, int nz, bool kmajor, int R) {
    const uint64_t dims[3] = {(uint64_t)cols, (uint64_t)rows, (uint64_t)nz};
    const uint64_t str[2] = {(uint64_t)cols * 2, (uint64_t)rows * cols * 2};
    const uint32_t box[3] = {64, (uint32_t)(kmajor ? R : 64), 1};
    return make_tmap_bf16(m, p, 3, dims, str, box);
}
bool map_2d(CUtensorMap *m, const void *p, int cols, int rows, bool kmajor, int R) {
    const uint64_t dims[2] = {(uint64_t)cols, (uint64_t)rows};
    const uint64_t str[1] = {(uint64_t)cols * 2};
    const uint32_t box[2] = {64, (uint32_t)(kmajor ? R : 64)};
    return make_tmap_bf16(m, p, 2, dims, str, box);
}

Operand opnd(int mode, int kmajor, int zmul = 1, int zoff = 0, int mn_off = 0) {
    Operand o;
    o.mode = mode; o.kmajor = kmajor; o.zmul = zmul; o.zoff = zoff; o.mn_off = mn_off;
    return o;
}

Epi epi_base(int op, void *out, int out_mode, int out_f32, int ldo, int ncols_out, int out_rows = kC) {
    Epi e;
    memset(&e, 0, sizeof(e));
    e.op = op; e.out = out; e.out_mode = out_mode; e.out_f32 = out_f32; e.ldo = ldo; e.ncols_out = ncols_out;
    e.out_rows = out_rows; e.out_zmul = 1; e.out_zoff = 0; e.scale = 1.f; e.rot_sign = 1;
    return e;
}

static int bwd_sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        n <= 0)
        return 152;
    return n;
}

cudaError_t gemm(const BwdGeo &g, int mtiles, int N, const CUtensorMap &a0, const Operand &A0, const CUtensorMap &b0,
                 const Operand &B0, int K0, const CUtensorMap *a1, const Operand *A1, const CUtensorMap *b1,
                 const Operand *B1, int K1, const Epi &e, cudaStream_t st) {
    GemmArgs ga;
    memset(&ga, 0, sizeof(ga));
    ga.nterms = a1 ? 2 : 1;
    ga.t[0].A = A0; ga.t[0].B = B0; ga.t[0].K = K0;
    if (a1) { ga.t[1].A = *A1; ga.t[1].B = *B1; ga.t[1].K = K1; }
    ga.N = N; ga.BH = g.BH; ga.L = g.L; ga.nchunks = g.nch; ga.e = e;
    ga.err = device_error_word();
    const size_t stage = (size_t)kC * 64 * 2 + (size_t)N * 64 * 2;
    int stages = (int)((100 * 1024) / stage);
    if (stages > kMaxStages) stages = kMaxStages;
    if (stages < 2) stages = 2;
    const int smem = (int)(stages * stage + 256 + 1024);
    cudaError_t err = cudaFuncSetAttribute(k_bgemm, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (err != cudaSuccess) return err;
    // persistent grid: as many CTAs as fit on the device at once (shared memory and TMEM: 2N
    // columns each), at most one per tile
    const int ntiles = g.Z * mtiles;
    int per_sm = (int)((227 * 1024) / smem);
    const int cols = N <= 16 ? 32 : N <= 32 ? 64 : N <= 64 ? 128 : N <= 128 ? 256 : 512;
    if (per_sm > 512 / cols) per_sm = 512 / cols;
    if (per_sm < 1) per_sm = 1;
    int nblk = bwd_sm_count() * per_sm;
    if (nblk > ntiles) nblk = ntiles;
    ProfScope ps(BLA_K_BWD, st);
    k_bgemm<<<nblk, kThreads, smem, st>>>(a0, b0, a1 ? *a1 : a0, b1 ? *b1 : b0, ga, stages, ntiles);
    return cudaGetLastError();
}

}  // namespace

const char *bwd_unsupported(const OpDims &d) {
    if (d.dtype != BLA_BF16) return "the backward is implemented for bf16 tensors";
    return fwd_bf16_unsupported(d);
}

size_t bwd_workspace_bytes(const OpDims &d) {
    if (bwd_unsupported(d)) return 0;
    BwdGeo g = bwd_geo(d);
    return bwd_ws(d, g).total;
}

cudaError_t bwd_run(const OpDims &d, const void *q, const void *k, const void *v, const void *o, const void *dout,
                    const float *lse, void *dq, void *dk, void *dv, void *workspace, cudaStream_t st) {
    BwdGeo g = bwd_geo(d);
    if (g.L == 0) return cudaSuccess;
    BwdWs w = bwd_ws(d, g);
    char *ws = static_cast<char *>(workspace);
    Tables t;
    tables_carve(d, kC, ws + w.tables, &t);
    cudaError_t e = tables_build(d, t, st);
    if (e != cudaSuccess) return e;
    bf16 *eb = reinterpret_cast<bf16 *>(ws + w.eb), *phi = reinterpret_cast<bf16 *>(ws + w.phi);
    if ((e = build_bf16_tables(d, g.RP, g.SP, eb, phi, st)) != cudaSuccess) return e;
    float *cphase = nullptr;
    if (d.absolute) {
        cphase = reinterpret_cast<float *>(ws + w.cphase);
        const int n = g.nch * g.M;
        ProfScope ps(BLA_K_BWD, st);
        k_chunk_phase<<<(n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024, 256, 0, st>>>(g.M, g.nch, d.w, cphase);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    float *cb = reinterpret_cast<float *>(ws + w.cb), *dKi = reinterpret_cast<float *>(ws + w.dKi);
    float *dVi = reinterpret_cast<float *>(ws + w.dVi), *dl = reinterpret_cast<float *>(ws + w.dl);
    bf16 *wb = reinterpret_cast<bf16 *>(ws + w.wb), *lb = reinterpret_cast<bf16 *>(ws + w.lb);
    bf16 *Pb = reinterpret_cast<bf16 *>(ws + w.P), *Yb = reinterpret_cast<bf16 *>(ws + w.Y);
    bf16 *pb = reinterpret_cast<bf16 *>(ws + w.p), *Ab = reinterpret_cast<bf16 *>(ws + w.A);
    bf16 *Gb = reinterpret_cast<bf16 *>(ws + w.G), *dGb = reinterpret_cast<bf16 *>(ws + w.dG);
    bf16 *dUb = reinterpret_cast<bf16 *>(ws + w.dU), *dsb = reinterpret_cast<bf16 *>(ws + w.ds);
    bf16 *dXb = reinterpret_cast<bf16 *>(ws + w.dX), *dPb = reinterpret_cast<bf16 *>(ws + w.dP);
    const int D = g.D, R2 = g.R2, S = g.S, SP = g.SP, Z = g.Z;
    const int rt = g.R2 <= 128 ? 1 : g.R2 / 128;   // 128-row tiles of an [R2 x D] result

    // ---- tensor maps
    CUtensorMap qK, qM, kK, kM, vK, vM, dOK, dOM, ebK128, ebKR, ebM, phiK, phiM;
    CUtensorMap wbK, wbM, lbM, PK, YK, pK, AK, AM, GK, GM, dGK, dUK, dsK, dXK, dXM, dPK, dPM;
    bool ok = map_seq(&qK, q, g, D, true, kC) && map_seq(&qM, q, g, D, false, 0) && map_seq(&kK, k, g, D, true, kC) &&
              map_seq(&kM, k, g, D, false, 0) && map_seq(&vK, v, g, D, true, kC) && map_seq(&vM, v, g, D, false, 0) &&
              map_seq(&dOK, dout, g, D, true, kC) && map_seq(&dOM, dout, g, D, false, 0) &&
              map_2d(&ebK128, eb, kC, g.RP, true, 128) && map_2d(&ebKR, eb, kC, g.RP, true, R2) &&
              map_2d(&ebM, eb, kC, g.RP, false, 0) && map_2d(&phiK, phi, R2, SP, true, S) &&
              map_2d(&phiM, phi, R2, SP, false, 0) && map_z(&wbK, wb, D, R2, 2 * Z, true, R2) &&
              map_z(&wbM, wb, D, R2, 2 * Z, false, 0) && map_z(&lbM, lb, D, R2, 2 * Z, false, 0) &&
              map_z(&PK, Pb, kC, kC, Z, true, kC) && map_z(&YK, Yb, R2, kC, Z, true, kC) &&
              map_z(&pK, pb, SP, kC, Z, true, kC) && map_z(&AK, Ab, R2, kC, Z, true, kC) &&
              map_z(&AM, Ab, R2, kC, Z, false, 0) && map_z(&GK, Gb, kC, kC, Z, true, kC) &&
              map_z(&GM, Gb, kC, kC, Z, false, 0) && map_z(&dGK, dGb, kC, kC, Z, true, kC) &&
              map_z(&dUK, dUb, R2, kC, Z, true, kC) && map_z(&dsK, dsb, SP, kC, Z, true, kC) &&
              map_z(&dXK, dXb, R2, kC, Z, true, kC) && map_z(&dXM, dXb, R2, kC, Z, false, 0) &&
              map_z(&dPK, dPb, kC, kC, Z, true, kC) && map_z(&dPM, dPb, kC, kC, Z, false, 0);
    (void)GK;
    if (!ok) return cudaErrorInvalidValue;
    const Operand SEQK = opnd(OP_SEQ, 1), SEQM = opnd(OP_SEQ, 0);
    const Operand ZK = opnd(OP_Z, 1), ZM = opnd(OP_Z, 0);
    const Operand SHK = opnd(OP_SHARED, 1), SHM = opnd(OP_SHARED, 0);
    const Operand WK_K = opnd(OP_Z, 1, 2, 0), WV_K = opnd(OP_Z, 1, 2, 1);
    const Operand WK_M = opnd(OP_Z, 0, 2, 0), LK_M = opnd(OP_Z, 0, 2, 0), LV_M = opnd(OP_Z, 0, 2, 1);

    // ---- 0. forward chunk states: contrib = EB X_c, then the scan
    for (int x = 0; x < 2; ++x) {
        Epi ep = epi_base(EP_PLAIN, cb, OUT_Z, 1, D, D, R2);
        ep.out_zmul = 2; ep.out_zoff = x;
        // A = EB (rows r, K = tau'), B = X_c MN-major (K rows tau', N = d)
        if ((e = gemm(g, rt, D, ebK128, SHK, x ? vM : kM, SEQM, kC, nullptr, nullptr, nullptr, nullptr, 0, ep, st)) !=
            cudaSuccess)
            return e;
    }
    {
        long long total = (long long)g.BH * 2 * g.M * D;
        int blocks = (int)((total + 255) / 256);
        if (blocks > 4096) blocks = 4096;
        ProfScope ps(BLA_K_BWD, st);
        k_state_scan<<<blocks, 256, 0, st>>>(g.BH, g.nch, g.M, D, t.erel, cb, wb, 0);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    Epi ep;
    // ---- 1. recompute the chunk's forward quantities
    ep = epi_base(EP_CAUSAL, Pb, OUT_Z, 0, kC, kC);                                   // P = tril(Q K^T)
    if ((e = gemm(g, 1, kC, qK, SEQK, kK, SEQK, D, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_ROT, Yb, OUT_Z, 0, R2, R2); ep.erel = t.erel; ep.cphase = cphase; ep.M = g.M;         // Y = rot+(P EB^T + Q W_K^T)
    if ((e = gemm(g, 1, R2, PK, ZK, ebKR, SHK, kC, &qK, &SEQK, &wbK, &WK_K, D, ep, st))) return e;
    ep = epi_base(EP_PROB, pb, OUT_Z, 0, SP, SP);                                      // p from lse
    ep.scale = d.scale; ep.lse = lse; ep.delta = t.delta; ep.S = S;
    if ((e = gemm(g, 1, S, YK, ZK, phiK, SHK, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_ROT, Ab, OUT_Z, 0, R2, R2); ep.erel = t.erel; ep.cphase = cphase; ep.M = g.M; ep.rot_sign = -1;   // A' = rot-(p PHI)
    if ((e = gemm(g, 1, R2, pK, ZK, phiM, SHM, SP, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_CAUSAL, Gb, OUT_Z, 0, kC, kC);                                   // G = tril(A' EB)
    if ((e = gemm(g, 1, kC, AK, ZK, ebM, SHM, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    // ---- 2. local adjoints
    ep = epi_base(EP_CAUSAL, dGb, OUT_Z, 0, kC, kC);                                  // dG = tril(dO V^T)
    if ((e = gemm(g, 1, kC, dOK, SEQK, vK, SEQK, D, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_ROT, dUb, OUT_Z, 0, R2, R2); ep.erel = t.erel; ep.cphase = cphase; ep.M = g.M;        // dU = rot+(dG EB^T + dO W_V^T)
    if ((e = gemm(g, 1, R2, dGK, ZK, ebKR, SHK, kC, &dOK, &SEQK, &wbK, &WV_K, D, ep, st))) return e;
    {
        long long total = (long long)Z * kC;
        int blocks = (int)((total + 7) / 8);   // eight rows (warps) per block
        if (blocks > 16384) blocks = 16384;
        ProfScope ps(BLA_K_BWD, st);
        k_rowdot<<<blocks, 256, 0, st>>>(g.BH, g.L, g.nch, D, (const bf16 *)dout, (const bf16 *)o, dl);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    ep = epi_base(EP_DS, dsb, OUT_Z, 0, SP, SP); ep.pbuf = pb; ep.ldp = SP; ep.dl = dl;  // ds = p (dU PHI^T - dl)
    if ((e = gemm(g, 1, S, dUK, ZK, phiK, SHK, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_ROT, dXb, OUT_Z, 0, R2, R2); ep.erel = t.erel; ep.cphase = cphase; ep.M = g.M;        // dX = rot-(scale ds PHI)
    ep.rot_sign = -1; ep.scale = d.scale;
    if ((e = gemm(g, 1, R2, dsK, ZK, phiM, SHM, SP, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_CAUSAL, dPb, OUT_Z, 0, kC, kC);                                  // dP = tril(dX EB)
    if ((e = gemm(g, 1, kC, dXK, ZK, ebM, SHM, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_PLAIN, dq, OUT_SEQ, 0, D, D);                                     // dQ = dP K + dX W_K
    if ((e = gemm(g, 1, D, dPK, ZK, kM, SEQM, kC, &dXK, &ZK, &wbM, &WK_M, R2, ep, st))) return e;
    ep = epi_base(EP_PLAIN, dKi, OUT_Z, 1, D, D);                                      // dK intra = dP^T Q
    if ((e = gemm(g, 1, D, dPM, ZM, qM, SEQM, kC, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_PLAIN, dVi, OUT_Z, 1, D, D);                                      // dV intra = G^T dO
    if ((e = gemm(g, 1, D, GM, ZM, dOM, SEQM, kC, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_PLAIN, cb, OUT_Z, 1, D, D, R2); ep.out_zmul = 2; ep.out_zoff = 0;   // contrib K = dX^T Q
    if ((e = gemm(g, rt, D, dXM, ZM, qM, SEQM, kC, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_PLAIN, cb, OUT_Z, 1, D, D, R2); ep.out_zmul = 2; ep.out_zoff = 1;   // contrib V = A'^T dO
    if ((e = gemm(g, rt, D, AM, ZM, dOM, SEQM, kC, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    // ---- 3. adjoint states, backwards over the chunks
    {
        long long total = (long long)g.BH * 2 * g.M * D;
        int blocks = (int)((total + 255) / 256);
        if (blocks > 4096) blocks = 4096;
        ProfScope ps(BLA_K_BWD, st);
        k_state_scan<<<blocks, 256, 0, st>>>(g.BH, g.nch, g.M, D, t.erel, cb, lb, 1);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    // ---- 4. dK = dK intra + EB^T Lk, dV = dV intra + EB^T Lv
    ep = epi_base(EP_ADD, dk, OUT_SEQ, 0, D, D); ep.addend = dKi;
    if ((e = gemm(g, 1, D, ebM, SHM, lbM, LK_M, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    ep = epi_base(EP_ADD, dv, OUT_SEQ, 0, D, D); ep.addend = dVi;
    if ((e = gemm(g, 1, D, ebM, SHM, lbM, LV_M, R2, nullptr, nullptr, nullptr, nullptr, 0, ep, st))) return e;
    return cudaSuccess;
}

}  // namespace bla
