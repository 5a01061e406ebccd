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
// The chunk-local contractions run on the tensor cores through one batched kernel, k_bgemm: a
// persistent CTA walks (chunk, 128-row tile) tiles and computes sum_t A_t B_t (up to two terms)
// with A, B streamed by TMA in 64-wide K blocks through a shared-memory ring, accumulates in TMEM
// and applies a fused epilogue (causal mask, per-mode phase rotation, probability recompute from
// lse, dS).  The states run through two chunk-sequential kernels, one CTA per (head, K or V):
// k_fwd_states rebuilds the forward's chunk states, k_adj_states carries the adjoint states
// backwards and writes dK and dV on the way; both keep the state in registers and take each
// chunk's contribution from the tensor cores.
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
enum EpiOp { EP_PLAIN = 0, EP_CAUSAL, EP_ROT, EP_PROB, EP_DS };
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

// ------------------------------------------------------------------ chunk-sequential state kernels
//
// One CTA per (head, x) with x = 0 (K) or 1 (V) walks the chunks in order and keeps the fp32 state
// in the registers of its eight epilogue warps (thread = state row r, warpgroup wg = columns
// [wg D/2, (wg+1) D/2)); the tensor cores compute each chunk's contribution into TMEM.
//   k_fwd_states  W_0 = 0, W_{c+1} = rot_C (W_c + EB X_c): the forward's chunk states (bf16, every c)
//   k_adj_states  L_last = 0, L_{c-1} = rot_C^T (L_c + X_c^T), X_c^T = dX^T Q (K) or A'^T dO (V),
//                 and the gradient dK_c = dP^T Q + EB^T L_c (K) or dV_c = G^T dO + EB^T L_c (V)
// Warps 0-7 are the epilogue, 8 issues TMA loads, 9 allocates TMEM and issues the MMAs.

constexpr int kSeqThreads = 320;
constexpr int kSeqEpiWarps = 8;

// SW128 descriptors of the chunk kernels' tiles.  A K-major tile stores [K/64][rows][64] (row =
// M or N index); an MN-major tile stores [MN/64][krows][64] (row = K index).
__device__ __forceinline__ uint64_t seq_kmaj(uint32_t base, int rows, int blk, int k) {
    return tc::sdesc_sw128(base + (uint32_t)((k >> 2) * rows * 128 + blk * 128 * 128 + (k & 3) * 32), 16, 1024);
}
__device__ __forceinline__ uint64_t seq_mnmaj(uint32_t base, int krows, int blk, int k) {
    return tc::sdesc_sw128(base + (uint32_t)(blk * 2 * krows * 128 + k * 16 * 128), (uint32_t)krows * 128u, 1024);
}

// 64 (or 32) bf16 values of one row into global memory (16-byte stores).
template <int N>
__device__ __forceinline__ void st_row_global(bf16 *dst, const float *v) {
#pragma unroll
    for (int i = 0; i < N; i += 8)
        *reinterpret_cast<uint4 *>(dst + i) =
            make_uint4(tc::pack_bf16x2(v[i], v[i + 1]), tc::pack_bf16x2(v[i + 2], v[i + 3]),
                       tc::pack_bf16x2(v[i + 4], v[i + 5]), tc::pack_bf16x2(v[i + 6], v[i + 7]));
}

// One step of rot_C (sign +1) or its transpose (sign -1) on interleaved (Re, Im) rows held by
// lane pairs (2m, 2m+1) of a warp.
template <int N>
__device__ __forceinline__ void rot_rows(float (&s)[N], bool odd, float cs, float sn, float sign) {
    const float sg = sign * sn;
#pragma unroll
    for (int i = 0; i < N; ++i) {
        const float partner = __shfl_xor_sync(0xffffffffu, s[i], 1);
        s[i] = odd ? fmaf(sg, partner, cs * s[i]) : fmaf(-sg, partner, cs * s[i]);
    }
}

// 32 values of one row of a [cols/64][rows_per_block][64] bf16 tile in the 128-byte-swizzled layout.
__device__ __forceinline__ void st_row32_bf16_seq(uint8_t *tile, int rows_per_block, int row, int col0, const float *v) {
    uint8_t *blk = tile + (size_t)(col0 >> 6) * rows_per_block * 128;
    const int c = col0 & 63;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 pk;
        pk.x = tc::pack_bf16x2(v[q * 8 + 0], v[q * 8 + 1]);
        pk.y = tc::pack_bf16x2(v[q * 8 + 2], v[q * 8 + 3]);
        pk.z = tc::pack_bf16x2(v[q * 8 + 4], v[q * 8 + 5]);
        pk.w = tc::pack_bf16x2(v[q * 8 + 6], v[q * 8 + 7]);
        *reinterpret_cast<uint4 *>(blk + tc::sw128_offset(row, c + q * 8)) = pk;
    }
}

struct SeqArgs {
    int BH, L, nch, M, R2, RP, D;
    const float *erel;   // (cos, sin)(m w tau), [C+1][M][2]
    bf16 *wout;          // k_fwd_states: [BH][nch][2][R2][D]
    bf16 *gout[2];       // k_adj_states: dk, dv [BH][L][D]
    int *err;
};

enum FsBar { FS_EB, FS_FULL0, FS_EMPTY0 = FS_FULL0 + 4, FS_DFULL0 = FS_EMPTY0 + 4, FS_DEMPTY0 = FS_DFULL0 + 2,
             FS_COUNT = FS_DEMPTY0 + 2 };
constexpr int kFsStages = 3;

// The chunk states W_c leave through shared memory: the eight epilogue warps write their rows into a
// staging tile ([D/64][RP rows][64], 128-byte swizzled; two tiles when they fit) and thread 0 stores it
// by TMA, instead of every thread storing its own row (32 rows per warp store, half-filled sectors).
template <int NB>
struct FsStaging {
    static constexpr int buffers = NB == 1 ? 2 : 1;
};

template <int D, int NB>
__global__ void __launch_bounds__(kSeqThreads, 1)
    k_fwd_states(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                 const __grid_constant__ CUtensorMap tm_eb, const __grid_constant__ CUtensorMap tm_w, SeqArgs a) {
    constexpr int DH = D / 2, RP = NB * 128;
    constexpr int SBUF = FsStaging<NB>::buffers, w_bytes = RP * D * 2;
    const int x = blockIdx.x & 1, bh = blockIdx.x >> 1;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sEB = sm;                                   // [2][RP][64] K-major A (rows r, K = u)
    uint8_t *sX = sEB + RP * 256;                        // kFsStages x [D/64][128 u][64] MN-major B
    constexpr int x_bytes = 128 * D * 2;
    uint8_t *sWst = sX + kFsStages * x_bytes;            // SBUF x [D/64][RP][64]: W_c staging
    uint64_t *bar = reinterpret_cast<uint64_t *>(sWst + SBUF * w_bytes);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + FS_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + FS_COUNT + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nupd = a.nch - 1;                          // chunks whose contribution is needed

    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[FS_EB], 1);
        for (int i = 0; i < kFsStages; ++i) { tc::mbar_init(&bar[FS_FULL0 + i], 1); tc::mbar_init(&bar[FS_EMPTY0 + i], 1); }
        for (int i = 0; i < 2; ++i) { tc::mbar_init(&bar[FS_DFULL0 + i], 1); tc::mbar_init(&bar[FS_DEMPTY0 + i], kSeqEpiWarps); }
        ctl->abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, 512); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;
    tc::pdl_wait();      // the tables

    if (warp == 8) {
        if (lane == 0 && nupd > 0) {
            const CUtensorMap *mx = x ? &tm_v : &tm_k;
            tc::mbar_arrive_expect_tx(&bar[FS_EB], (uint32_t)(RP * 256));
            for (int b = 0; b < NB; ++b)
                for (int ub = 0; ub < 2; ++ub)
                    tc::tma_load_2d(sEB + ub * RP * 128 + b * 128 * 128, &tm_eb, &bar[FS_EB], ub * 64, b * 128);
            uint32_t ph[kFsStages] = {0, 0, 0};
            for (int c = 0; c < nupd && !ctl->abort; ++c) {
                const int st = c % kFsStages;
                if (c >= kFsStages && !wait_bar(&bar[FS_EMPTY0 + st], ph[st], ctl, a.err, 10)) break;
                tc::mbar_arrive_expect_tx(&bar[FS_FULL0 + st], (uint32_t)x_bytes);
                for (int db = 0; db < D / 64; ++db)
                    tc::tma_load_3d(sX + st * x_bytes + db * 128 * 128, mx, &bar[FS_FULL0 + st], db * 64, c * kC, bh);
            }
        }
    } else if (warp == 9) {
        if (lane == 0 && nupd > 0) {
            uint32_t ph_eb = 0, ph[kFsStages] = {0, 0, 0}, ph_de[2] = {0, 0};
            const uint32_t idesc = tc::idesc_bf16(128, D, false, true);
            bool ok = wait_bar(&bar[FS_EB], ph_eb, ctl, a.err, 11);
            for (int c = 0; c < nupd && ok; ++c) {
                const int st = c % kFsStages, buf = c & 1;
                if (c >= 2 && !wait_bar(&bar[FS_DEMPTY0 + buf], ph_de[buf], ctl, a.err, 12)) break;
                if (!wait_bar(&bar[FS_FULL0 + st], ph[st], ctl, a.err, 13)) break;
                tc::tc_fence_after();
                const uint32_t xs = tc::smem_u32(sX + st * x_bytes), es = tc::smem_u32(sEB);
                for (int b = 0; b < NB; ++b)
                    for (int k = 0; k < 8; ++k)
                        tc::mma_bf16(tb + (uint32_t)((buf * NB + b) * D), seq_kmaj(es, RP, b, k), seq_mnmaj(xs, 128, 0, k),
                                     idesc, k > 0 ? 1u : 0u);
                tc::mma_commit(&bar[FS_EMPTY0 + st]);
                tc::mma_commit(&bar[FS_DFULL0 + buf]);
            }
        }
    } else {
        const int wg = warp >> 2, lane_base = (warp & 3) * 32, row = lane_base + lane;
        const bool odd = row & 1;
        float s[NB][DH];
        float cs[NB], sn[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int m = (b * 128 + row) >> 1;
            cs[b] = m < a.M ? a.erel[((size_t)kC * a.M + m) * 2] : 1.f;
            sn[b] = m < a.M ? a.erel[((size_t)kC * a.M + m) * 2 + 1] : 0.f;
#pragma unroll
            for (int i = 0; i < DH; ++i) s[b][i] = 0.f;
        }
        uint32_t ph_df[2] = {0, 0};
        for (int c = 0; c < a.nch; ++c) {
            // W_c, by thread 0's TMA store of the staging tile (the one two chunks back has been read)
            uint8_t *stile = sWst + (SBUF == 2 ? (c & 1) : 0) * w_bytes;
            if (threadIdx.x == 0) {
                if (SBUF == 2) tc::bulk_wait_read1();
                else tc::bulk_wait_read0();
            }
            tc::named_bar(1, kSeqEpiWarps * 32);
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const int r = b * 128 + row;
                if (r < a.R2) {
#pragma unroll
                    for (int g0 = 0; g0 < DH; g0 += 32) st_row32_bf16_seq(stile, RP, r, wg * DH + g0, s[b] + g0);
                }
            }
            tc::fence_proxy_async_smem();
            tc::named_bar(1, kSeqEpiWarps * 32);
            if (threadIdx.x == 0) {
                for (int db = 0; db < D / 64; ++db)
                    tc::tma_store_3d(&tm_w, stile + db * RP * 128, db * 64, 0, (bh * a.nch + c) * 2 + x);
                tc::bulk_commit();
            }
            if (c == nupd) break;
            const int buf = c & 1;
            if (!wait_bar(&bar[FS_DFULL0 + buf], ph_df[buf], ctl, a.err, 14)) break;
            tc::tc_fence_after();
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                float v[DH];
                tc::tmem_ld<DH>(tb + ((uint32_t)lane_base << 16) + (uint32_t)((buf * NB + b) * D + wg * DH), v);
#pragma unroll
                for (int i = 0; i < DH; ++i) s[b][i] += v[i];
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[FS_DEMPTY0 + buf]);
#pragma unroll
            for (int b = 0; b < NB; ++b) rot_rows<DH>(s[b], odd, cs[b], sn[b], 1.f);
        }
        if (threadIdx.x == 0) tc::bulk_wait0();
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, 512);
    }
}

enum AsBar { AS_EB, AS_FULL0, AS_FREE0 = AS_FULL0 + 2, AS_CFULL0 = AS_FREE0 + 2, AS_CEMPTY0 = AS_CFULL0 + 2,
             AS_LB = AS_CEMPTY0 + 2, AS_DKFULL, AS_DKEMPTY, AS_COUNT };

// Shared memory of k_adj_states: EB, then `stages` x (Xa [RP/64][128 t][64], Bq [D/64][128 t][64],
// Pa [2][128 t][64]); L_c (bf16, [D/64][R2][64]) is written over the stage's Xa once its MMA is done,
// and the chunk's dK or dV rows over its Pa once the gradient MMAs are done.  Thread 0 stores those
// rows by TMA and releases the stage to the producer once the store has read them.
__host__ __device__ inline int adj_stage_bytes(int RP, int D) { return RP * 256 + D * 256 + 2 * 128 * 128; }

template <int D, int NB>
__global__ void __launch_bounds__(kSeqThreads, 1)
    k_adj_states(const __grid_constant__ CUtensorMap tm_dx, const __grid_constant__ CUtensorMap tm_ap,
                 const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_do,
                 const __grid_constant__ CUtensorMap tm_dp, const __grid_constant__ CUtensorMap tm_g,
                 const __grid_constant__ CUtensorMap tm_eb, const __grid_constant__ CUtensorMap tm_gk,
                 const __grid_constant__ CUtensorMap tm_gv, SeqArgs a, int stages) {
    constexpr int DH = D / 2, RP = NB * 128;
    constexpr int NCB = NB == 1 ? 2 : 1;                 // contribution buffers in TMEM
    const int x = blockIdx.x & 1, bh = blockIdx.x >> 1;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sEB = sm;                                   // [2][RP][64]: MN-major A of EB^T (M = u, K = r)
    uint8_t *sStage = sEB + RP * 256;
    const int sbytes = adj_stage_bytes(RP, D);
    uint64_t *bar = reinterpret_cast<uint64_t *>(sStage + stages * sbytes);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + AS_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + AS_COUNT + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = a.nch, R2 = a.R2;
    const uint32_t colDK = (uint32_t)(NCB * NB * D);
    // chunk i of the walk is c = nch - 1 - i

    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[AS_EB], 1);
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&bar[AS_FULL0 + i], 1);
            tc::mbar_init(&bar[AS_FREE0 + i], 1);
            tc::mbar_init(&bar[AS_CFULL0 + i], 1);
            tc::mbar_init(&bar[AS_CEMPTY0 + i], kSeqEpiWarps);
        }
        tc::mbar_init(&bar[AS_LB], kSeqEpiWarps);
        tc::mbar_init(&bar[AS_DKFULL], 1);
        tc::mbar_init(&bar[AS_DKEMPTY], kSeqEpiWarps);
        ctl->abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, 512); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;
    tc::pdl_wait();      // the chains' outputs

    if (warp == 8) {
        if (lane == 0) {
            const CUtensorMap *ma = x ? &tm_ap : &tm_dx, *mb = x ? &tm_do : &tm_q, *mp = x ? &tm_g : &tm_dp;
            tc::mbar_arrive_expect_tx(&bar[AS_EB], (uint32_t)(RP * 256));
            for (int b = 0; b < NB; ++b)
                for (int ub = 0; ub < 2; ++ub)
                    tc::tma_load_2d(sEB + ub * RP * 128 + b * 128 * 128, &tm_eb, &bar[AS_EB], ub * 64, b * 128);
            uint32_t ph[2] = {0, 0};
            for (int i = 0; i < nch && !ctl->abort; ++i) {
                const int c = nch - 1 - i, st = i % stages;
                if (i >= stages && !wait_bar(&bar[AS_FREE0 + st], ph[st], ctl, a.err, 20)) break;
                uint8_t *base = sStage + st * sbytes;
                tc::mbar_arrive_expect_tx(&bar[AS_FULL0 + st], (uint32_t)sbytes);
                const int z = bh * nch + c;
                for (int rb = 0; rb < RP / 64; ++rb)            // beyond R2: zero fill
                    tc::tma_load_3d(base + rb * 128 * 128, ma, &bar[AS_FULL0 + st], rb * 64, 0, z);
                for (int db = 0; db < D / 64; ++db)
                    tc::tma_load_3d(base + RP * 256 + db * 128 * 128, mb, &bar[AS_FULL0 + st], db * 64, c * kC, bh);
                for (int ub = 0; ub < 2; ++ub)
                    tc::tma_load_3d(base + RP * 256 + D * 256 + ub * 128 * 128, mp, &bar[AS_FULL0 + st], ub * 64, 0, z);
                // the chunk `stages` steps later into L2 now: with at most `stages` 96 KB stages in shared
                // memory the loads alone would keep too few bytes in flight
                if (i + stages < nch) {
                    const int cn = c - stages, zn = bh * nch + cn;
                    for (int rb = 0; rb < RP / 64; ++rb) tc::tma_prefetch_3d(ma, rb * 64, 0, zn);
                    for (int db = 0; db < D / 64; ++db) tc::tma_prefetch_3d(mb, db * 64, cn * kC, bh);
                    for (int ub = 0; ub < 2; ++ub) tc::tma_prefetch_3d(mp, ub * 64, 0, zn);
                }
            }
        }
    } else if (warp == 9) {
        if (lane == 0) {
            uint32_t ph_eb = 0, ph[2] = {0, 0}, ph_ce[2] = {0, 0}, ph_lb = 0, ph_dke = 0;
            const uint32_t id_c = tc::idesc_bf16(128, D, true, true);   // A = (dX or A')^T, B = Q or dO: MN-major
            bool ok = wait_bar(&bar[AS_EB], ph_eb, ctl, a.err, 21);
            for (int i = 0; i < nch && ok; ++i) {
                ok = false;
                const int st = i % stages, cb = i % NCB;
                if (!wait_bar(&bar[AS_FULL0 + st], ph[st], ctl, a.err, 22)) break;
                if (i >= NCB && !wait_bar(&bar[AS_CEMPTY0 + cb], ph_ce[cb], ctl, a.err, 23)) break;
                tc::tc_fence_after();
                const uint32_t base = tc::smem_u32(sStage + st * sbytes);
                const uint32_t xa = base, bq = base + RP * 256, pa = bq + D * 256, es = tc::smem_u32(sEB);
                // X_c^T = (dX or A')^T (Q or dO): M = state rows, K = the chunk's tokens
                for (int b = 0; b < NB; ++b)
                    for (int k = 0; k < 8; ++k)
                        tc::mma_bf16(tb + (uint32_t)((cb * NB + b) * D), seq_mnmaj(xa, 128, b, k), seq_mnmaj(bq, 128, 0, k),
                                     id_c, k > 0 ? 1u : 0u);
                tc::mma_commit(&bar[AS_CFULL0 + cb]);
                // dK_c = dP^T Q + EB^T L_c (or dV_c = G^T dO + EB^T L_c): M = the chunk's tokens u
                if (i > 0 && !wait_bar(&bar[AS_DKEMPTY], ph_dke, ctl, a.err, 24)) break;
                tc::tc_fence_after();
                for (int k = 0; k < 8; ++k)
                    tc::mma_bf16(tb + colDK, seq_mnmaj(pa, 128, 0, k), seq_mnmaj(bq, 128, 0, k), id_c, k > 0 ? 1u : 0u);
                if (!wait_bar(&bar[AS_LB], ph_lb, ctl, a.err, 25)) break;
                tc::tc_fence_after();
                for (int k = 0; k < R2 / 16; ++k)
                    tc::mma_bf16(tb + colDK, seq_mnmaj(es, RP, 0, k), seq_mnmaj(xa, R2, 0, k), id_c, 1u);
                tc::mma_commit(&bar[AS_DKFULL]);   // (the epilogue releases the stage after the dK store)
                ok = true;
            }
        }
    } else {
        const int wg = warp >> 2, lane_base = (warp & 3) * 32, row = lane_base + lane;
        const bool odd = row & 1;
        float s[NB][DH];
        float cs[NB], sn[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int m = (b * 128 + row) >> 1;
            cs[b] = m < a.M ? a.erel[((size_t)kC * a.M + m) * 2] : 1.f;
            sn[b] = m < a.M ? a.erel[((size_t)kC * a.M + m) * 2 + 1] : 0.f;
#pragma unroll
            for (int i = 0; i < DH; ++i) s[b][i] = 0.f;
        }
        uint32_t ph_cf[2] = {0, 0}, ph_dkf = 0;
        const CUtensorMap *tg = x ? &tm_gv : &tm_gk;
        for (int i = 0; i < nch; ++i) {
            const int c = nch - 1 - i, st = i % stages, cb = i % NCB;
            // L_c (bf16) over the stage's Xa once the contribution MMA has read it
            if (!wait_bar(&bar[AS_CFULL0 + cb], ph_cf[cb], ctl, a.err, 26)) break;
            tc::tc_fence_after();
            uint8_t *lb = sStage + st * sbytes;
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const int r = b * 128 + row;
                if (r < R2) {
#pragma unroll
                    for (int g0 = 0; g0 < DH; g0 += 32) st_row32_bf16_seq(lb, R2, r, wg * DH + g0, s[b] + g0);
                }
            }
            tc::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[AS_LB]);
            // L_{c-1} = rot_C^T (L_c + X_c^T)
            if (c > 0) {
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    float v[DH];
                    tc::tmem_ld<DH>(tb + ((uint32_t)lane_base << 16) + (uint32_t)((cb * NB + b) * D + wg * DH), v);
#pragma unroll
                    for (int j = 0; j < DH; ++j) s[b][j] += v[j];
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[AS_CEMPTY0 + cb]);
            if (c > 0) {
#pragma unroll
                for (int b = 0; b < NB; ++b) rot_rows<DH>(s[b], odd, cs[b], sn[b], -1.f);
            }
            // the chunk's gradient rows, staged over the stage's dP / G tile (its MMAs are done) and
            // stored by thread 0 (rows past L are clipped by the tensor map)
            if (!wait_bar(&bar[AS_DKFULL], ph_dkf, ctl, a.err, 27)) break;
            tc::tc_fence_after();
            uint8_t *gt = sStage + st * sbytes + RP * 256 + D * 256;
            {
                float v[DH];
                tc::tmem_ld<DH>(tb + ((uint32_t)lane_base << 16) + colDK + (uint32_t)(wg * DH), v);
#pragma unroll
                for (int g0 = 0; g0 < DH; g0 += 32) st_row32_bf16_seq(gt, 128, row, wg * DH + g0, v + g0);
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[AS_DKEMPTY]);
            tc::fence_proxy_async_smem();
            tc::named_bar(1, kSeqEpiWarps * 32);
            if (threadIdx.x == 0) {
                for (int db = 0; db < D / 64; ++db) tc::tma_store_3d(tg, gt + db * 128 * 128, db * 64, c * kC, bh);
                tc::bulk_commit();
                // a stage goes back to the producer once its rows are read: with two stages the previous
                // step's (this step's store may still be reading), with one this step's own
                if (stages == 1) {
                    tc::bulk_wait_read0();
                    tc::mbar_arrive(&bar[AS_FREE0]);
                } else if (i > 0) {
                    tc::bulk_wait_read1();
                    tc::mbar_arrive(&bar[AS_FREE0 + (i - 1) % stages]);
                }
            }
        }
        if (threadIdx.x == 0) tc::bulk_wait0();
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, 512);
    }
}

// ------------------------------------------------------------------ fused chunk chains
//
// For 2M <= 128 and S <= 64 the chunk-local part of the backward runs as two persistent kernels,
// one CTA per SM walking chunks, whose intermediates stay on chip (TMEM accumulators drained into
// bf16 shared-memory tiles that feed the next MMA):
//   k_chain_fwd  P = tril(Q K^T) -> Y = rot+(P EB^T + Q W_K^T) -> p -> A' = rot-(p PHI) -> G = tril(A' EB)
//                writes p, A' and G
//   k_chain_adj  dG = tril(dO V^T) -> dU = rot+(dG EB^T + dO W_V^T) -> ds = p (dU PHI^T - rowsum(dO o))
//                -> dX = rot-(scale ds PHI) -> dP = tril(dX EB) -> dQ = dP K + dX W_K
//                writes dX, dP and dQ
// Shared-memory tiles are 128B-swizzled [cols/64][rows][64]: K-major when rows index M or N, and
// the same bytes serve as an MN-major B operand whose K index is the row (EB, PHI, K, W).
// Warps 0-7 drain TMEM in 32-column chunks (warpgroup wg takes chunks wg, wg + 2, ...), warp 8
// issues TMA loads, warp 9 issues the MMAs.  Outputs are written as bf16 tiles in shared memory
// and stored by TMA (thread 0 issues the stores after an epilogue barrier, and waits for them to
// have read their tiles before the next chunk overwrites any tile).

struct ChainArgs {
    int BH, L, nch, Z, M, R2, S, SP, D;
    float scale;
    const float *erel;    // (cos, sin)(m w tau), [C+1][M][2]
    const float *cphase;  // absolute form: (cos, sin)(-m w c C), [nch][M][2]; else null
    const float *lse;     // [BH][L]
    const int *delta;     // [S]
    const bf16 *o;        // [BH][L][D]
    int *err;
};

// Phases of one thread's column range in a chunk: e^{i m0 w tau} for its first mode m0 and the step
// e^{i w tau} between consecutive modes (tau = the row's offset in the chunk), or in the absolute
// form the chunk's e^{-i m0 w t0} and e^{-i w t0}.
struct RotPh {
    float c0, s0, c1, s1;
};

__device__ __forceinline__ RotPh chain_phases(const ChainArgs &a, int c, int row, int m0) {
    const float *ptab = a.cphase ? a.cphase + (size_t)c * a.M * 2 : a.erel + (size_t)row * a.M * 2;
    RotPh r;
    r.c0 = __ldg(ptab + m0 * 2);
    r.s0 = __ldg(ptab + m0 * 2 + 1);
    r.c1 = __ldg(ptab + 2);
    r.s1 = __ldg(ptab + 3);
    return r;
}

// Rotation of N interleaved (Re, Im) columns by the phases of `ph` (sign +1) or their transposes
// (sign -1), times `scale`.
template <int N>
__device__ __forceinline__ void chain_rot(float (&v)[N], const RotPh &ph, float sign, float scale) {
    float cs = ph.c0, sn = ph.s0;
#pragma unroll
    for (int i = 0; i < N; i += 2) {
        const float sg = sign * sn, xr = v[i], xi = v[i + 1];
        v[i] = scale * (cs * xr - sg * xi);
        v[i + 1] = scale * (sg * xr + cs * xi);
        const float t = cs * ph.c1 - sn * ph.s1;
        sn = sn * ph.c1 + cs * ph.s1;
        cs = t;
    }
}

template <int N>
__device__ __forceinline__ void chain_causal(float (&v)[N], int row, int col0) {
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (col0 + i > row) v[i] = 0.f;
}

template <int N>
__device__ __forceinline__ void st_tile_row(uint8_t *tile, int row, int col0, const float (&v)[N]) {
#pragma unroll
    for (int g = 0; g < N; g += 32) st_row32_bf16_seq(tile, 128, row, col0 + g, v + g);
}

__device__ __forceinline__ uint32_t tm_addr(uint32_t tb, int lane_base, int col) {
    return tb + ((uint32_t)lane_base << 16) + (uint32_t)col;
}

// ---- k_chain_fwd
enum CfBar { CF_TAB, CF_IN_FULL, CF_IN_FREE, CF_ACC1, CF_ACC2, CF_ACC3, CF_ACC4, CF_ACC5, CF_T1, CF_T2, CF_SP, CF_A,
             CF_ESYNC, CF_COUNT };

struct ChainLayout {
    int eb, phi, t0, t1, t2, t3, t4, sp, bars, total;
};

// k_chain_fwd: t0 = Q, t1 = K, t2 = W_K, t3 = T1 (P, then A'), t4 = T2 (Y, then G), sp = p.
// k_chain_adj: t0 = dO, t1 = V then K, t2 = W_V then W_K, t3 = T1 (dG, then dP), t4 = T2 (dU, then
//              dX, then dQ), sp = p, then ds.
// The last 1 KB holds the barriers, the slot lags and the rows' rowsum(dO o).
__host__ __device__ inline ChainLayout chain_layout(int R2, int S, int SP, int D) {
    ChainLayout l;
    int off = 0;
    l.eb = off;  off += R2 * 256;
    l.phi = off; off += R2 * S * 2;
    off = (off + 1023) & ~1023;
    l.t0 = off;  off += 256 * D;
    l.t1 = off;  off += 256 * D;
    l.t2 = off;  off += R2 * D * 2;
    l.t3 = off;  off += 128 * 256;
    l.t4 = off;  off += 128 * 256;
    l.sp = off;  off += SP * 256;
    l.bars = off; off += 1024;
    l.total = off;
    return l;
}

template <int R2, int S, int D>
__global__ void __launch_bounds__(kSeqThreads, 1)
    k_chain_fwd(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_eb,
                const __grid_constant__ CUtensorMap tm_phi, const __grid_constant__ CUtensorMap tm_po,
                const __grid_constant__ CUtensorMap tm_ao, const __grid_constant__ CUtensorMap tm_go, ChainArgs a) {
    constexpr int SP = S < 64 ? 64 : S, HX = R2 / 2, HS = S >= 64 ? S / 2 : S;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const ChainLayout lay = chain_layout(R2, S, SP, D);
    uint8_t *sEB = sm + lay.eb, *sPHI = sm + lay.phi, *sQ = sm + lay.t0, *sK = sm + lay.t1, *sW = sm + lay.t2;
    uint8_t *sT1 = sm + lay.t3, *sT2 = sm + lay.t4, *sP = sm + lay.sp;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + lay.bars);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + CF_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + CF_COUNT + 1);
    int *sdelta = reinterpret_cast<int *>(bar + CF_COUNT + 2);   // [S]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int colP = 0, colX = 128, colS = 0, colU = 0, colG = 128;   // s after P is drained; U after s

    if (threadIdx.x == 0) {
        for (int i = 0; i < CF_COUNT; ++i) {
            const bool epi = i == CF_T1 || i == CF_T2 || i == CF_SP || i == CF_A || i == CF_ESYNC;
            tc::mbar_init(&bar[i], epi ? kSeqEpiWarps : 1);
        }
        ctl->abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, 256); tc::tmem_relinquish(); }
    tc::pdl_wait();      // the chunk states and the tables
    for (int j = threadIdx.x; j < S; j += blockDim.x) sdelta[j] = a.delta[j];
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;

    if (warp == 8) {
        if (lane == 0) {
            tc::mbar_arrive_expect_tx(&bar[CF_TAB], (uint32_t)(R2 * 256 + R2 * S * 2));
            for (int ub = 0; ub < 2; ++ub) tc::tma_load_2d(sEB + ub * R2 * 128, &tm_eb, &bar[CF_TAB], ub * 64, 0);
            for (int rb = 0; rb < R2 / 64; ++rb) tc::tma_load_2d(sPHI + rb * S * 128, &tm_phi, &bar[CF_TAB], rb * 64, 0);
            uint32_t ph_free = 0;
            for (int z = blockIdx.x, i = 0; z < a.Z && !ctl->abort; z += gridDim.x, ++i) {
                const int bh = z / a.nch, c = z % a.nch;
                if (i > 0 && !wait_bar(&bar[CF_IN_FREE], ph_free, ctl, a.err, 30)) break;
                tc::mbar_arrive_expect_tx(&bar[CF_IN_FULL], (uint32_t)(2 * 256 * D + R2 * D * 2));
                for (int db = 0; db < D / 64; ++db) {
                    tc::tma_load_3d(sQ + db * 128 * 128, &tm_q, &bar[CF_IN_FULL], db * 64, c * kC, bh);
                    tc::tma_load_3d(sK + db * 128 * 128, &tm_k, &bar[CF_IN_FULL], db * 64, c * kC, bh);
                    tc::tma_load_3d(sW + db * R2 * 128, &tm_w, &bar[CF_IN_FULL], db * 64, 0, 2 * z);
                }
            }
        }
    } else if (warp == 9) {
        if (lane == 0) {
            uint32_t ph[CF_COUNT] = {};
            constexpr uint32_t id_P = tc::idesc_bf16(128, 128, false, false), id_X = tc::idesc_bf16(128, R2, false, false);
            constexpr uint32_t id_S = tc::idesc_bf16(128, S, false, false), id_U = tc::idesc_bf16(128, R2, false, true);
            constexpr uint32_t id_G = tc::idesc_bf16(128, 128, false, true);
            const uint32_t q = tc::smem_u32(sQ), k = tc::smem_u32(sK), w = tc::smem_u32(sW), eb = tc::smem_u32(sEB);
            const uint32_t phi = tc::smem_u32(sPHI), t1 = tc::smem_u32(sT1), t2 = tc::smem_u32(sT2), sp = tc::smem_u32(sP);
            bool ok = wait_bar(&bar[CF_TAB], ph[CF_TAB], ctl, a.err, 31);
            // P = Q K^T of a chunk, into region 0 (free once the previous chunk's A' has been drained)
            auto issue_p = [&]() -> bool {
                if (!wait_bar(&bar[CF_IN_FULL], ph[CF_IN_FULL], ctl, a.err, 32)) return false;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma_bf16(tb + colP, seq_kmaj(q, 128, 0, kk), seq_kmaj(k, 128, 0, kk), id_P, kk > 0);
                tc::mma_commit(&bar[CF_ACC1]);
                return true;
            };
            ok = ok && (int)blockIdx.x < a.Z && issue_p();
            for (int z = blockIdx.x; z < a.Z && ok; z += gridDim.x) {
                ok = false;
                if (!wait_bar(&bar[CF_T1], ph[CF_T1], ctl, a.err, 34)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)                      // X = P EB^T + Q W_K^T
                    tc::mma_bf16(tb + colX, seq_kmaj(t1, 128, 0, kk), seq_kmaj(eb, R2, 0, kk), id_X, kk > 0);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma_bf16(tb + colX, seq_kmaj(q, 128, 0, kk), seq_kmaj(w, R2, 0, kk), id_X, 1u);
                tc::mma_commit(&bar[CF_ACC2]);
                tc::mma_commit(&bar[CF_IN_FREE]);
                if (!wait_bar(&bar[CF_T2], ph[CF_T2], ctl, a.err, 35)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < R2 / 16; ++kk)                // s = Y PHI^T
                    tc::mma_bf16(tb + colS, seq_kmaj(t2, 128, 0, kk), seq_kmaj(phi, S, 0, kk), id_S, kk > 0);
                tc::mma_commit(&bar[CF_ACC3]);
                if (!wait_bar(&bar[CF_SP], ph[CF_SP], ctl, a.err, 36)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < S / 16; ++kk)                 // U = p PHI
                    tc::mma_bf16(tb + colU, seq_kmaj(sp, 128, 0, kk), seq_mnmaj(phi, S, 0, kk), id_U, kk > 0);
                tc::mma_commit(&bar[CF_ACC4]);
                if (!wait_bar(&bar[CF_A], ph[CF_A], ctl, a.err, 37)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < R2 / 16; ++kk)                // G = A' EB
                    tc::mma_bf16(tb + colG, seq_kmaj(t1, 128, 0, kk), seq_mnmaj(eb, R2, 0, kk), id_G, kk > 0);
                tc::mma_commit(&bar[CF_ACC5]);
                // the next chunk's P runs while G is drained: region 0 held U, drained before A' arrived
                ok = z + (int)gridDim.x >= a.Z || issue_p();
            }
        }
    } else {
        // warpgroup wg drains columns [wg N/2, (wg+1) N/2) of each N-column result (N = S = 32: wg 0 only)
        const int wg = warp >> 2, lane_base = (warp & 3) * 32, row = lane_base + lane;
        uint32_t ph[CF_COUNT] = {};
        auto arrive = [&](int b) {
            tc::fence_proxy_async_smem();
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[b]);
        };
        auto esync = [&](int which) -> bool {
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[CF_ESYNC]);
            return wait_bar(&bar[CF_ESYNC], ph[CF_ESYNC], ctl, a.err, which);
        };
        for (int z = blockIdx.x; z < a.Z; z += gridDim.x) {
            const int bh = z / a.nch, c = z % a.nch, t = c * kC + row;
            const bool live = t < a.L;
            const float lse = live ? __ldg(a.lse + (size_t)bh * a.L + t) : 0.f;
            const RotPh rp = chain_phases(a, c, row, wg * HX / 2);
            // the previous chunk's stores must have read their tiles
            if (threadIdx.x == 0) tc::bulk_wait_read0();
            if (!esync(45)) break;
            // P = tril(Q K^T)
            if (!wait_bar(&bar[CF_ACC1], ph[CF_ACC1], ctl, a.err, 40)) break;
            tc::tc_fence_after();
            {
                float v[64];
                tc::tmem_ld<64>(tm_addr(tb, lane_base, colP + wg * 64), v);
                chain_causal<64>(v, row, wg * 64);
                st_tile_row<64>(sT1, row, wg * 64, v);
            }
            arrive(CF_T1);
            // Y = rot+(X)
            if (!wait_bar(&bar[CF_ACC2], ph[CF_ACC2], ctl, a.err, 41)) break;
            tc::tc_fence_after();
            {
                float v[HX];
                tc::tmem_ld<HX>(tm_addr(tb, lane_base, colX + wg * HX), v);
                chain_rot<HX>(v, rp, 1.f, 1.f);
                st_tile_row<HX>(sT2, row, wg * HX, v);
            }
            arrive(CF_T2);
            // p = exp(scale s - lse), masked; slots beyond S are zero
            if (!wait_bar(&bar[CF_ACC3], ph[CF_ACC3], ctl, a.err, 42)) break;
            tc::tc_fence_after();
            if (S >= 64 || wg == 0) {
                float v[HS];
                tc::tmem_ld<HS>(tm_addr(tb, lane_base, colS + wg * HS), v);
#pragma unroll
                for (int j = 0; j < HS; ++j) {
                    const int jj = wg * HS + j;
                    v[j] = (live && t >= sdelta[jj]) ? __expf(a.scale * v[j] - lse) : 0.f;
                }
                st_tile_row<HS>(sP, row, wg * HS, v);
            } else {
                float v[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = 0.f;
                st_tile_row<32>(sP, row, 32, v);
            }
            tc::fence_proxy_async_smem();
            if (!esync(46)) break;
            if (threadIdx.x == 0) {
                for (int jb = 0; jb < SP / 64; ++jb) tc::tma_store_3d(&tm_po, sP + jb * 128 * 128, jb * 64, 0, z);
                tc::bulk_commit();
            }
            arrive(CF_SP);
            // A' = rot-(p PHI)
            if (!wait_bar(&bar[CF_ACC4], ph[CF_ACC4], ctl, a.err, 43)) break;
            tc::tc_fence_after();
            {
                float v[HX];
                tc::tmem_ld<HX>(tm_addr(tb, lane_base, colU + wg * HX), v);
                chain_rot<HX>(v, rp, -1.f, 1.f);
                st_tile_row<HX>(sT1, row, wg * HX, v);
            }
            tc::fence_proxy_async_smem();
            if (!esync(47)) break;
            if (threadIdx.x == 0) {
                for (int rb = 0; rb < R2 / 64; ++rb) tc::tma_store_3d(&tm_ao, sT1 + rb * 128 * 128, rb * 64, 0, z);
                tc::bulk_commit();
            }
            arrive(CF_A);
            // G = tril(A' EB), staged in the Y tile (read by s long before)
            if (!wait_bar(&bar[CF_ACC5], ph[CF_ACC5], ctl, a.err, 44)) break;
            tc::tc_fence_after();
            {
                float v[64];
                tc::tmem_ld<64>(tm_addr(tb, lane_base, colG + wg * 64), v);
                chain_causal<64>(v, row, wg * 64);
                st_tile_row<64>(sT2, row, wg * 64, v);
            }
            tc::fence_proxy_async_smem();
            if (!esync(48)) break;
            if (threadIdx.x == 0) {
                for (int ub = 0; ub < 2; ++ub) tc::tma_store_3d(&tm_go, sT2 + ub * 128 * 128, ub * 64, 0, z);
                tc::bulk_commit();
            }
            __syncwarp();
        }
        if (threadIdx.x == 0) tc::bulk_wait0();
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, 256);
    }
}

// ---- k_chain_adj
// Loads: dO and p of chunk c+1 go in as soon as chunk c has consumed its own (dU and rowsum(dO o);
// ds PHI), V and W_V once dQ is done; K and W_K replace V and W_V after dU.
enum CaBar { CA_TAB, CA_DO_FULL, CA_P_FULL, CA_VW_FULL, CA_VW_FREE, CA_SP_FREE, CA_KW_FULL, CA_KW_FREE, CA_ACC1,
             CA_ACC2, CA_ACC3, CA_ACC4, CA_ACC5, CA_ACC6, CA_T1, CA_T2, CA_DS, CA_DX, CA_DP, CA_TFREE, CA_ESYNC,
             CA_COUNT };

template <int R2, int S, int D>
__global__ void __launch_bounds__(kSeqThreads, 1)
    k_chain_adj(const __grid_constant__ CUtensorMap tm_do, const __grid_constant__ CUtensorMap tm_v,
                const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_w,
                const __grid_constant__ CUtensorMap tm_p, const __grid_constant__ CUtensorMap tm_eb,
                const __grid_constant__ CUtensorMap tm_phi, const __grid_constant__ CUtensorMap tm_dxo,
                const __grid_constant__ CUtensorMap tm_dpo, const __grid_constant__ CUtensorMap tm_dqo, ChainArgs a) {
    constexpr int SP = S < 64 ? 64 : S, HX = R2 / 2, HS = S >= 64 ? S / 2 : S, HD = D / 2;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const ChainLayout lay = chain_layout(R2, S, SP, D);
    uint8_t *sEB = sm + lay.eb, *sPHI = sm + lay.phi, *sDO = sm + lay.t0, *sVK = sm + lay.t1, *sWW = sm + lay.t2;
    uint8_t *sT1 = sm + lay.t3, *sT2 = sm + lay.t4, *sP = sm + lay.sp;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + lay.bars);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + CA_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + CA_COUNT + 1);
    float *sdl = reinterpret_cast<float *>(bar + CA_COUNT + 2);   // [128] rowsum(dO o)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int colA = 0, colB = 128, colC = 256, colD = 384;

    if (threadIdx.x == 0) {
        for (int i = 0; i < CA_COUNT; ++i) {
            const bool epi = i == CA_T1 || i == CA_T2 || i == CA_DS || i == CA_DX || i == CA_DP || i == CA_TFREE ||
                             i == CA_ESYNC;
            tc::mbar_init(&bar[i], i == CA_VW_FREE ? 1 + kSeqEpiWarps : (epi ? kSeqEpiWarps : 1));
        }
        ctl->abort = 0;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, 512); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;
    tc::pdl_wait();      // p and the chunk states

    if (warp == 8) {
        if (lane == 0) {
            tc::mbar_arrive_expect_tx(&bar[CA_TAB], (uint32_t)(R2 * 256 + R2 * S * 2));
            for (int ub = 0; ub < 2; ++ub) tc::tma_load_2d(sEB + ub * R2 * 128, &tm_eb, &bar[CA_TAB], ub * 64, 0);
            for (int rb = 0; rb < R2 / 64; ++rb) tc::tma_load_2d(sPHI + rb * S * 128, &tm_phi, &bar[CA_TAB], rb * 64, 0);
            uint32_t ph_kwf = 0, ph_vwf = 0, ph_spf = 0;
            auto load_do = [&](int z) {
                const int bh = z / a.nch, c = z % a.nch;
                tc::mbar_arrive_expect_tx(&bar[CA_DO_FULL], (uint32_t)(256 * D));
                for (int db = 0; db < D / 64; ++db)
                    tc::tma_load_3d(sDO + db * 128 * 128, &tm_do, &bar[CA_DO_FULL], db * 64, c * kC, bh);
            };
            auto load_p = [&](int z) {
                tc::mbar_arrive_expect_tx(&bar[CA_P_FULL], (uint32_t)(SP * 256));
                for (int jb = 0; jb < SP / 64; ++jb)
                    tc::tma_load_3d(sP + jb * 128 * 128, &tm_p, &bar[CA_P_FULL], jb * 64, 0, z);
            };
            auto load_vw = [&](int z) {
                const int bh = z / a.nch, c = z % a.nch;
                tc::mbar_arrive_expect_tx(&bar[CA_VW_FULL], (uint32_t)(256 * D + R2 * D * 2));
                for (int db = 0; db < D / 64; ++db) {
                    tc::tma_load_3d(sVK + db * 128 * 128, &tm_v, &bar[CA_VW_FULL], db * 64, c * kC, bh);
                    tc::tma_load_3d(sWW + db * R2 * 128, &tm_w, &bar[CA_VW_FULL], db * 64, 0, 2 * z + 1);
                }
            };
            auto load_kw = [&](int z) {
                const int bh = z / a.nch, c = z % a.nch;
                tc::mbar_arrive_expect_tx(&bar[CA_KW_FULL], (uint32_t)(256 * D + R2 * D * 2));
                for (int db = 0; db < D / 64; ++db) {
                    tc::tma_load_3d(sVK + db * 128 * 128, &tm_k, &bar[CA_KW_FULL], db * 64, c * kC, bh);
                    tc::tma_load_3d(sWW + db * R2 * 128, &tm_w, &bar[CA_KW_FULL], db * 64, 0, 2 * z);
                }
            };
            const int z0 = blockIdx.x;
            if (z0 < a.Z) { load_do(z0); load_p(z0); load_vw(z0); }
            for (int z = z0; z < a.Z && !ctl->abort; z += gridDim.x) {
                const int zn = z + (int)gridDim.x;
                // chunk z has read V, W_V and dO: its K, W_K, and the next chunk's dO
                if (!wait_bar(&bar[CA_VW_FREE], ph_vwf, ctl, a.err, 51)) break;
                load_kw(z);
                if (zn < a.Z) {
                    load_do(zn);
                    // the next chunk's o (for rowsum(dO o)) into L2
                    const int nbh = zn / a.nch, nc = zn % a.nch, rows = min(kC, a.L - nc * kC);
                    tc::bulk_prefetch_l2(a.o + ((size_t)nbh * a.L + (size_t)nc * kC) * D, (uint32_t)(rows * D * 2));
                }
                if (zn >= a.Z) break;
                // chunk z's ds has been read: the next chunk's p
                if (!wait_bar(&bar[CA_SP_FREE], ph_spf, ctl, a.err, 52)) break;
                load_p(zn);
                // chunk z's dQ is done: the next chunk's V and W_V
                if (!wait_bar(&bar[CA_KW_FREE], ph_kwf, ctl, a.err, 50)) break;
                load_vw(zn);
            }
        }
    } else if (warp == 9) {
        if (lane == 0) {
            uint32_t ph[CA_COUNT] = {};
            constexpr uint32_t id_G = tc::idesc_bf16(128, 128, false, false), id_U = tc::idesc_bf16(128, R2, false, false);
            constexpr uint32_t id_S = tc::idesc_bf16(128, S, false, false), id_X = tc::idesc_bf16(128, R2, false, true);
            constexpr uint32_t id_P = tc::idesc_bf16(128, 128, false, true), id_Q = tc::idesc_bf16(128, D, false, true);
            const uint32_t dO = tc::smem_u32(sDO), vk = tc::smem_u32(sVK), ww = tc::smem_u32(sWW), eb = tc::smem_u32(sEB);
            const uint32_t phi = tc::smem_u32(sPHI), t1 = tc::smem_u32(sT1), t2 = tc::smem_u32(sT2), sp = tc::smem_u32(sP);
            bool ok = wait_bar(&bar[CA_TAB], ph[CA_TAB], ctl, a.err, 52);
            for (int z = blockIdx.x, i = 0; z < a.Z && ok; z += gridDim.x, ++i) {
                ok = false;
                if (!wait_bar(&bar[CA_DO_FULL], ph[CA_DO_FULL], ctl, a.err, 53)) break;
                if (!wait_bar(&bar[CA_VW_FULL], ph[CA_VW_FULL], ctl, a.err, 74)) break;
                if (i > 0 && !wait_bar(&bar[CA_TFREE], ph[CA_TFREE], ctl, a.err, 54)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)                 // dG = dO V^T
                    tc::mma_bf16(tb + colA, seq_kmaj(dO, 128, 0, kk), seq_kmaj(vk, 128, 0, kk), id_G, kk > 0);
                tc::mma_commit(&bar[CA_ACC1]);
                if (!wait_bar(&bar[CA_T1], ph[CA_T1], ctl, a.err, 55)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)                      // dU = dG EB^T + dO W_V^T
                    tc::mma_bf16(tb + colB, seq_kmaj(t1, 128, 0, kk), seq_kmaj(eb, R2, 0, kk), id_U, kk > 0);
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma_bf16(tb + colB, seq_kmaj(dO, 128, 0, kk), seq_kmaj(ww, R2, 0, kk), id_U, 1u);
                tc::mma_commit(&bar[CA_ACC2]);
                tc::mma_commit(&bar[CA_VW_FREE]);
                if (!wait_bar(&bar[CA_T2], ph[CA_T2], ctl, a.err, 56)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < R2 / 16; ++kk)                // dp = dU PHI^T
                    tc::mma_bf16(tb + colC, seq_kmaj(t2, 128, 0, kk), seq_kmaj(phi, S, 0, kk), id_S, kk > 0);
                tc::mma_commit(&bar[CA_ACC3]);
                if (!wait_bar(&bar[CA_DS], ph[CA_DS], ctl, a.err, 57)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < S / 16; ++kk)                 // ds PHI
                    tc::mma_bf16(tb + colA, seq_kmaj(sp, 128, 0, kk), seq_mnmaj(phi, S, 0, kk), id_X, kk > 0);
                tc::mma_commit(&bar[CA_ACC4]);
                tc::mma_commit(&bar[CA_SP_FREE]);
                if (!wait_bar(&bar[CA_DX], ph[CA_DX], ctl, a.err, 58)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < R2 / 16; ++kk)                // dP = dX EB
                    tc::mma_bf16(tb + colB, seq_kmaj(t2, 128, 0, kk), seq_mnmaj(eb, R2, 0, kk), id_P, kk > 0);
                tc::mma_commit(&bar[CA_ACC5]);
                if (!wait_bar(&bar[CA_DP], ph[CA_DP], ctl, a.err, 59)) break;
                if (!wait_bar(&bar[CA_KW_FULL], ph[CA_KW_FULL], ctl, a.err, 60)) break;
                tc::tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)                      // dQ = dP K + dX W_K
                    tc::mma_bf16(tb + colD, seq_kmaj(t1, 128, 0, kk), seq_mnmaj(vk, 128, 0, kk), id_Q, kk > 0);
#pragma unroll
                for (int kk = 0; kk < R2 / 16; ++kk)
                    tc::mma_bf16(tb + colD, seq_kmaj(t2, 128, 0, kk), seq_mnmaj(ww, R2, 0, kk), id_Q, 1u);
                tc::mma_commit(&bar[CA_ACC6]);
                tc::mma_commit(&bar[CA_KW_FREE]);
                ok = true;
            }
        }
    } else {
        const int wg = warp >> 2, lane_base = (warp & 3) * 32, row = lane_base + lane;
        uint32_t ph[CA_COUNT] = {};
        auto arrive = [&](int b) {
            tc::fence_proxy_async_smem();
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[b]);
        };
        auto esync = [&](int which) -> bool {
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[CA_ESYNC]);
            return wait_bar(&bar[CA_ESYNC], ph[CA_ESYNC], ctl, a.err, which);
        };
        constexpr int LPR = D / 8;            // lanes per row in the rowsum (8 bf16 each)
        constexpr int RPI = 32 / LPR;         // rows per warp iteration
        for (int z = blockIdx.x; z < a.Z; z += gridDim.x) {
            const int bh = z / a.nch, c = z % a.nch;
            const RotPh rp = chain_phases(a, c, row, wg * HX / 2);
            if (threadIdx.x == 0) tc::bulk_wait_read0();
            if (!esync(68)) break;
            if (!wait_bar(&bar[CA_DO_FULL], ph[CA_DO_FULL], ctl, a.err, 61)) break;
            // rowsum(dO o) of 16 rows per warp, loads of o coalesced (LPR lanes per row); every load
            // is issued before the first is used
            {
                constexpr int NIT = 16 / RPI;
                const int d0 = (lane % LPR) * 8;
                uint4 ov[NIT];
#pragma unroll
                for (int it = 0; it < NIT; ++it) {
                    const int r = warp * 16 + it * RPI + lane / LPR, tt = c * kC + r;
                    ov[it] = tt < a.L ? __ldg(reinterpret_cast<const uint4 *>(a.o + ((size_t)bh * a.L + tt) * D + d0))
                                      : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int it = 0; it < NIT; ++it) {
                    const int r = warp * 16 + it * RPI + lane / LPR;
                    const uint4 gv = *reinterpret_cast<const uint4 *>(sDO + (d0 >> 6) * 128 * 128 + tc::sw128_offset(r, d0 & 63));
                    const uint32_t ow[4] = {ov[it].x, ov[it].y, ov[it].z, ov[it].w}, gw[4] = {gv.x, gv.y, gv.z, gv.w};
                    float acc = 0.f;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&ow[q]));
                        const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&gw[q]));
                        acc = fmaf(x.x, y.x, fmaf(x.y, y.y, acc));
                    }
#pragma unroll
                    for (int off = LPR / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
                    if (lane % LPR == 0) sdl[r] = acc;
                }
            }
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&bar[CA_VW_FREE]);
            if (!esync(73)) break;
            const float dl = sdl[row];
            // dG
            if (!wait_bar(&bar[CA_ACC1], ph[CA_ACC1], ctl, a.err, 62)) break;
            tc::tc_fence_after();
            {
                float v[64];
                tc::tmem_ld<64>(tm_addr(tb, lane_base, colA + wg * 64), v);
                chain_causal<64>(v, row, wg * 64);
                st_tile_row<64>(sT1, row, wg * 64, v);
            }
            arrive(CA_T1);
            // dU
            if (!wait_bar(&bar[CA_ACC2], ph[CA_ACC2], ctl, a.err, 63)) break;
            tc::tc_fence_after();
            {
                float v[HX];
                tc::tmem_ld<HX>(tm_addr(tb, lane_base, colB + wg * HX), v);
                chain_rot<HX>(v, rp, 1.f, 1.f);
                st_tile_row<HX>(sT2, row, wg * HX, v);
            }
            arrive(CA_T2);
            // ds = p (dp - dl), over p in place
            if (!wait_bar(&bar[CA_P_FULL], ph[CA_P_FULL], ctl, a.err, 75)) break;
            if (!wait_bar(&bar[CA_ACC3], ph[CA_ACC3], ctl, a.err, 64)) break;
            tc::tc_fence_after();
            if (S >= 64 || wg == 0) {
                float v[HS];
                tc::tmem_ld<HS>(tm_addr(tb, lane_base, colC + wg * HS), v);
#pragma unroll
                for (int g0 = 0; g0 < HS; g0 += 8) {
                    const int col = wg * HS + g0;
                    uint4 *pp = reinterpret_cast<uint4 *>(sP + (col >> 6) * 128 * 128 + tc::sw128_offset(row, col & 63));
                    const uint4 pk = *pp;
                    const uint32_t w[4] = {pk.x, pk.y, pk.z, pk.w};
                    uint32_t o4[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 pf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[e]));
                        o4[e] = tc::pack_bf16x2(pf.x * (v[g0 + 2 * e] - dl), pf.y * (v[g0 + 2 * e + 1] - dl));
                    }
                    *pp = make_uint4(o4[0], o4[1], o4[2], o4[3]);
                }
            }
            arrive(CA_DS);
            // dX = rot-(scale ds PHI)
            if (!wait_bar(&bar[CA_ACC4], ph[CA_ACC4], ctl, a.err, 65)) break;
            tc::tc_fence_after();
            {
                float v[HX];
                tc::tmem_ld<HX>(tm_addr(tb, lane_base, colA + wg * HX), v);
                chain_rot<HX>(v, rp, -1.f, a.scale);
                st_tile_row<HX>(sT2, row, wg * HX, v);
            }
            tc::fence_proxy_async_smem();
            if (!esync(69)) break;
            if (threadIdx.x == 0) {
                for (int rb = 0; rb < R2 / 64; ++rb) tc::tma_store_3d(&tm_dxo, sT2 + rb * 128 * 128, rb * 64, 0, z);
                tc::bulk_commit();
            }
            arrive(CA_DX);
            // dP = tril(dX EB)
            if (!wait_bar(&bar[CA_ACC5], ph[CA_ACC5], ctl, a.err, 66)) break;
            tc::tc_fence_after();
            {
                float v[64];
                tc::tmem_ld<64>(tm_addr(tb, lane_base, colB + wg * 64), v);
                chain_causal<64>(v, row, wg * 64);
                st_tile_row<64>(sT1, row, wg * 64, v);
            }
            tc::fence_proxy_async_smem();
            if (!esync(70)) break;
            if (threadIdx.x == 0) {
                for (int ub = 0; ub < 2; ++ub) tc::tma_store_3d(&tm_dpo, sT1 + ub * 128 * 128, ub * 64, 0, z);
                tc::bulk_commit();
            }
            arrive(CA_DP);
            // dQ, staged in the dX tile once dQ's MMA and dX's store have read it
            if (!wait_bar(&bar[CA_ACC6], ph[CA_ACC6], ctl, a.err, 67)) break;
            tc::tc_fence_after();
            float vq[HD];
            tc::tmem_ld<HD>(tm_addr(tb, lane_base, colD + wg * HD), vq);
            if (threadIdx.x == 0) tc::bulk_wait_read0();
            if (!esync(71)) break;
            st_tile_row<HD>(sT2, row, wg * HD, vq);
            tc::fence_proxy_async_smem();
            if (!esync(72)) break;
            if (threadIdx.x == 0) {
                for (int db = 0; db < D / 64; ++db) tc::tma_store_3d(&tm_dqo, sT2 + db * 128 * 128, db * 64, c * kC, bh);
                tc::bulk_commit();
            }
            arrive(CA_TFREE);
        }
        if (threadIdx.x == 0) tc::bulk_wait0();
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, 512);
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

// The fused chains hold their tiles in shared memory for 2M <= 128 and S <= 64.
bool chain_fits(const BwdGeo &g) { return g.R2 >= 64 && g.R2 <= 128 && g.S >= 32 && g.S <= 64; }

struct BwdWs {
    size_t tables, eb, phi, cphase, wb, P, Y, p, A, G, dG, dU, ds, dX, dP, dl, total;
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
    w.wb = take(2 * Z * 2 * g.R2 * g.D);
    // P, Y, dG, dU, ds and rowsum(dO o) go through memory only on the unfused route
    const size_t u = chain_fits(g) ? 0 : 1;
    w.P = take(u * 2 * Z * kC * kC);
    w.Y = take(u * 2 * Z * kC * g.R2);
    w.p = take(2 * Z * kC * g.SP);
    w.A = take(2 * Z * kC * g.R2);
    w.G = take(2 * Z * kC * kC);
    w.dG = take(u * 2 * Z * kC * kC);
    w.dU = take(u * 2 * Z * kC * g.R2);
    w.ds = take(u * 2 * Z * kC * g.SP);
    w.dX = take(2 * Z * kC * g.R2);
    w.dP = take(2 * Z * kC * kC);
    w.dl = take(u * 4 * Z * kC);
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

template <int D, int NB>
cudaError_t launch_fwd_states_t(const BwdGeo &g, const CUtensorMap &mk, const CUtensorMap &mv, const CUtensorMap &meb,
                                const CUtensorMap &mw, const SeqArgs &sa, cudaStream_t st) {
    // (both chunk kernels allocate all 512 TMEM columns: at least 120 KB of shared memory keeps a
    //  second CTA off the SM, so an allocation never waits for another CTA to finish)
    int smem = NB * 128 * 256 + kFsStages * 128 * D * 2 + FsStaging<NB>::buffers * NB * 128 * D * 2 + 256 + 1024;
    if (smem > 227 * 1024) return cudaErrorInvalidValue;
    if (smem < 120 * 1024) smem = 120 * 1024;
    cudaError_t e = cudaFuncSetAttribute(k_fwd_states<D, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_BWD, st);
    return launch_pdl(k_fwd_states<D, NB>, dim3(g.BH * 2), dim3(kSeqThreads), (size_t)smem, st, mk, mv, meb, mw, sa);
}

cudaError_t launch_fwd_states(const BwdGeo &g, const CUtensorMap &mk, const CUtensorMap &mv, const CUtensorMap &meb,
                              const CUtensorMap &mw, const SeqArgs &sa, cudaStream_t st) {
    const int NB = g.RP / 128;
    if (g.D == 128) return NB == 1 ? launch_fwd_states_t<128, 1>(g, mk, mv, meb, mw, sa, st)
                                   : launch_fwd_states_t<128, 2>(g, mk, mv, meb, mw, sa, st);
    if (g.D == 64) return NB == 1 ? launch_fwd_states_t<64, 1>(g, mk, mv, meb, mw, sa, st)
                                  : launch_fwd_states_t<64, 2>(g, mk, mv, meb, mw, sa, st);
    return cudaErrorInvalidValue;
}

template <int D, int NB>
cudaError_t launch_adj_states_t(const BwdGeo &g, const CUtensorMap &mdx, const CUtensorMap &map_, const CUtensorMap &mq,
                                const CUtensorMap &mdo, const CUtensorMap &mdp, const CUtensorMap &mg,
                                const CUtensorMap &meb, const CUtensorMap &mgk, const CUtensorMap &mgv,
                                const SeqArgs &sa, cudaStream_t st) {
    const int RP = NB * 128, sbytes = adj_stage_bytes(RP, D);
    int stages = (227 * 1024 - 1024 - 256 - RP * 256) / sbytes;
    if (stages > 2) stages = 2;
    if (stages < 1) return cudaErrorInvalidValue;
    int smem = RP * 256 + stages * sbytes + 256 + 1024;
    if (smem < 120 * 1024) smem = 120 * 1024;
    cudaError_t e = cudaFuncSetAttribute(k_adj_states<D, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_BWD, st);
    return launch_pdl(k_adj_states<D, NB>, dim3(g.BH * 2), dim3(kSeqThreads), (size_t)smem, st, mdx, map_, mq, mdo,
                      mdp, mg, meb, mgk, mgv, sa, stages);
}

cudaError_t launch_adj_states(const BwdGeo &g, const CUtensorMap &mdx, const CUtensorMap &map_, const CUtensorMap &mq,
                              const CUtensorMap &mdo, const CUtensorMap &mdp, const CUtensorMap &mg,
                              const CUtensorMap &meb, const CUtensorMap &mgk, const CUtensorMap &mgv, const SeqArgs &sa,
                              cudaStream_t st) {
    const int NB = g.RP / 128;
    if (g.D == 128) return NB == 1 ? launch_adj_states_t<128, 1>(g, mdx, map_, mq, mdo, mdp, mg, meb, mgk, mgv, sa, st)
                                   : launch_adj_states_t<128, 2>(g, mdx, map_, mq, mdo, mdp, mg, meb, mgk, mgv, sa, st);
    if (g.D == 64) return NB == 1 ? launch_adj_states_t<64, 1>(g, mdx, map_, mq, mdo, mdp, mg, meb, mgk, mgv, sa, st)
                                  : launch_adj_states_t<64, 2>(g, mdx, map_, mq, mdo, mdp, mg, meb, mgk, mgv, sa, st);
    return cudaErrorInvalidValue;
}

template <int R2, int S, int D>
cudaError_t launch_chains_t(const BwdGeo &g, const ChainArgs &ca, const CUtensorMap &mq, const CUtensorMap &mk,
                            const CUtensorMap &mv, const CUtensorMap &mdo, const CUtensorMap &mw, const CUtensorMap &mp,
                            const CUtensorMap &meb, const CUtensorMap &mphi, const CUtensorMap &ma,
                            const CUtensorMap &mg, const CUtensorMap &mdx, const CUtensorMap &mdp,
                            const CUtensorMap &mdq, cudaStream_t st) {
    const ChainLayout lay = chain_layout(R2, S, S < 64 ? 64 : S, D);
    const int smem = lay.total + 1024;
    cudaError_t e = cudaFuncSetAttribute(k_chain_fwd<R2, S, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_chain_adj<R2, S, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int nblk = bwd_sm_count();
    if (nblk > g.Z) nblk = g.Z;
    {
        ProfScope ps(BLA_K_BWD, st);
        e = launch_pdl(k_chain_fwd<R2, S, D>, dim3(nblk), dim3(kSeqThreads), (size_t)smem, st, mq, mk, mw, meb, mphi,
                       mp, ma, mg, ca);
    }
    if (e != cudaSuccess) return e;
    {
        ProfScope ps(BLA_K_BWD, st);
        e = launch_pdl(k_chain_adj<R2, S, D>, dim3(nblk), dim3(kSeqThreads), (size_t)smem, st, mdo, mv, mk, mw, mp,
                       meb, mphi, mdx, mdp, mdq, ca);
    }
    return e;
}

cudaError_t launch_chains(const BwdGeo &g, const ChainArgs &ca, const CUtensorMap &mq, const CUtensorMap &mk,
                          const CUtensorMap &mv, const CUtensorMap &mdo, const CUtensorMap &mw, const CUtensorMap &mp,
                          const CUtensorMap &meb, const CUtensorMap &mphi, const CUtensorMap &ma, const CUtensorMap &mg,
                          const CUtensorMap &mdx, const CUtensorMap &mdp, const CUtensorMap &mdq, cudaStream_t st) {
#define BLA_CHAIN(R, S_, D_)                                                                                          \
    if (g.R2 == R && g.S == S_ && g.D == D_)                                                                          \
        return launch_chains_t<R, S_, D_>(g, ca, mq, mk, mv, mdo, mw, mp, meb, mphi, ma, mg, mdx, mdp, mdq, st);
    BLA_CHAIN(64, 32, 64) BLA_CHAIN(64, 32, 128) BLA_CHAIN(64, 64, 64) BLA_CHAIN(64, 64, 128)
    BLA_CHAIN(128, 32, 64) BLA_CHAIN(128, 32, 128) BLA_CHAIN(128, 64, 64) BLA_CHAIN(128, 64, 128)
#undef BLA_CHAIN
    return cudaErrorInvalidValue;
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
    float *dl = reinterpret_cast<float *>(ws + w.dl);
    bf16 *wb = reinterpret_cast<bf16 *>(ws + w.wb);
    bf16 *Pb = reinterpret_cast<bf16 *>(ws + w.P), *Yb = reinterpret_cast<bf16 *>(ws + w.Y);
    bf16 *pb = reinterpret_cast<bf16 *>(ws + w.p), *Ab = reinterpret_cast<bf16 *>(ws + w.A);
    bf16 *Gb = reinterpret_cast<bf16 *>(ws + w.G), *dGb = reinterpret_cast<bf16 *>(ws + w.dG);
    bf16 *dUb = reinterpret_cast<bf16 *>(ws + w.dU), *dsb = reinterpret_cast<bf16 *>(ws + w.ds);
    bf16 *dXb = reinterpret_cast<bf16 *>(ws + w.dX), *dPb = reinterpret_cast<bf16 *>(ws + w.dP);
    const int D = g.D, R2 = g.R2, S = g.S, SP = g.SP, Z = g.Z;

    // ---- tensor maps
    CUtensorMap qK, kK, kM, vK, dOK, ebK128, ebKR, ebM, phiK, phiM;
    CUtensorMap wbK, wbM, PK, YK, pK, AK, GK, dGK, dUK, dsK, dXK, dPK, dkS, dvS;
    bool ok = map_seq(&qK, q, g, D, true, kC) && map_seq(&kK, k, g, D, true, kC) && map_seq(&kM, k, g, D, false, 0) &&
              map_seq(&vK, v, g, D, true, kC) && map_seq(&dOK, dout, g, D, true, kC) &&
              map_2d(&ebK128, eb, kC, g.RP, true, 128) && map_2d(&ebKR, eb, kC, g.RP, true, R2) &&
              map_2d(&ebM, eb, kC, g.RP, false, 0) && map_2d(&phiK, phi, R2, SP, true, S) &&
              map_2d(&phiM, phi, R2, SP, false, 0) && map_z(&wbK, wb, D, R2, 2 * Z, true, R2) &&
              map_z(&wbM, wb, D, R2, 2 * Z, false, 0) &&
              map_z(&PK, Pb, kC, kC, Z, true, kC) && map_z(&YK, Yb, R2, kC, Z, true, kC) &&
              map_z(&pK, pb, SP, kC, Z, true, kC) && map_z(&AK, Ab, R2, kC, Z, true, kC) &&
              map_z(&GK, Gb, kC, kC, Z, true, kC) && map_z(&dGK, dGb, kC, kC, Z, true, kC) &&
              map_z(&dUK, dUb, R2, kC, Z, true, kC) && map_z(&dsK, dsb, SP, kC, Z, true, kC) &&
              map_z(&dXK, dXb, R2, kC, Z, true, kC) && map_z(&dPK, dPb, kC, kC, Z, true, kC) &&
              map_seq(&dkS, dk, g, D, true, kC) && map_seq(&dvS, dv, g, D, true, kC);
    if (!ok) return cudaErrorInvalidValue;
    const Operand SEQK = opnd(OP_SEQ, 1), SEQM = opnd(OP_SEQ, 0);
    const Operand ZK = opnd(OP_Z, 1), ZM = opnd(OP_Z, 0);
    const Operand SHK = opnd(OP_SHARED, 1), SHM = opnd(OP_SHARED, 0);
    const Operand WK_K = opnd(OP_Z, 1, 2, 0), WV_K = opnd(OP_Z, 1, 2, 1);
    const Operand WK_M = opnd(OP_Z, 0, 2, 0);

    // ---- 0. forward chunk states W_c (bf16), scanned over the chunks of each head in registers
    SeqArgs sa;
    sa.BH = g.BH; sa.L = g.L; sa.nch = g.nch; sa.M = g.M; sa.R2 = R2; sa.RP = g.RP; sa.D = D;
    sa.erel = t.erel; sa.wout = wb; sa.gout[0] = static_cast<bf16 *>(dk); sa.gout[1] = static_cast<bf16 *>(dv);
    sa.err = device_error_word();
    if ((e = launch_fwd_states(g, kK, vK, ebK128, wbK, sa, st)) != cudaSuccess) return e;
    if (chain_fits(g)) {
        // ---- 1-2. the chunk-local chains, fused
        ChainArgs ca;
        ca.BH = g.BH; ca.L = g.L; ca.nch = g.nch; ca.Z = Z; ca.M = g.M; ca.R2 = R2; ca.S = S; ca.SP = SP; ca.D = D;
        ca.scale = d.scale; ca.erel = t.erel; ca.cphase = cphase; ca.lse = lse; ca.delta = t.delta;
        ca.o = static_cast<const bf16 *>(o);
        ca.err = sa.err;
        CUtensorMap dqK;
        if (!map_seq(&dqK, dq, g, D, true, kC)) return cudaErrorInvalidValue;
        if ((e = launch_chains(g, ca, qK, kK, vK, dOK, wbK, pK, ebKR, phiK, AK, GK, dXK, dPK, dqK, st)) != cudaSuccess)
            return e;
        if ((e = launch_adj_states(g, dXK, AK, qK, dOK, dPK, GK, ebK128, dkS, dvS, sa, st)) != cudaSuccess) return e;
        return cudaSuccess;
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
    // ---- 3. adjoint states backwards over the chunks, with dK = dP^T Q + EB^T Lk and
    //         dV = G^T dO + EB^T Lv for every chunk on the way
    if ((e = launch_adj_states(g, dXK, AK, qK, dOK, dPK, GK, ebK128, dkS, dvS, sa, st)) != cudaSuccess) return e;
    return cudaSuccess;
}

}  // namespace bla
