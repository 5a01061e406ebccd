// decay_chunk.cu -- the state-decayed forward (Sec. 3.3) in chunks of 64 tokens, bf16 operands.
//
// Per slot j the decayed state is a first-order linear recurrence,
//     X_j(t) = a_j(t) X_j(t-1) + D_j(t) x_t,     a_j(t) = 1 - D_j(t),  D_j(t) = D_M(t - Delta_j),
// for X = K~ (x = k) and X = V~ (x = v).  Over a chunk of C tokens starting at t0 (tau, u = 0..C-1
// the in-chunk positions) it unrolls to
//     X_j(t0 + tau) = A_j(tau) X_j(t0 - 1) + sum_{u <= tau} W_j(tau, u) x_{t0+u},
//     A_j(tau) = prod_{x <= tau} a_j(t0 + x),   W_j(tau, u) = D_j(t0 + u) prod_{u < x <= tau} a_j(t0 + x),
// so that, with P = Q_c K_c^T and Y = Q_c K~(t0-1)^T,
//     s[tau, j] = scale (A_j(tau) Y[tau, j] + sum_{u <= tau} P[tau, u] W_j(tau, u))       (Alg. 1 scores)
//     p = softmax over the slots with t >= Delta_j,
//     o = (p o A) V~(t0-1) + G V_c,   G[tau, u] = sum_j p[tau, j] W_j(tau, u)
//     X~(t0 + C - 1) = A_j(C-1) X~(t0 - 1) + Wend X_c,   Wend[j][u] = W_j(C-1, u).
// Every factor is a product of a's: nothing is divided, so the exact zeros of a (D = 1 at the
// kernel's peak) need no care.  The four contractions per chunk (P, Y, O and the state update) run
// on the tensor cores as warp-level bf16 MMAs with fp32 accumulation; the weighted triangle sums
// (s and G) run on the CUDA cores, walking u downward from tau with the running product r_j:
//     w = D_j(u) r,   r <- r a_j(u).
// The fp32 state lives in the MMA accumulator registers of the warps that update it; a bf16 copy
// in shared memory feeds the next chunk's Y and O.
//
// Parallelism: each head's sequence is cut into G segments.  Mode 0 (only when G > 1) runs every
// segment but the last from the zero state through the state updates alone and writes the
// segment's decay product prod a_j and its state delta; k_dchunk_scan chains them into the state
// entering each segment; mode 1 runs every segment from its entering state and writes o, lse and,
// from the last segment, the final state.
#include <math.h>

#include "decay.cuh"
#include "mma_sync.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace bla {

namespace {

using namespace wmma16;

constexpr int kDC = 64;            // tokens per chunk
constexpr int kDThreads = 512;     // 16 warps
constexpr int kDWarps = kDThreads / 32;
constexpr int kFS = kDC + 4;       // row stride (floats) of the fp32 [64][64] tiles

// ------------------------------------------------------------------ shared-memory layout

template <int D, int S>
struct DcLayout {
    static constexpr int kTile = kDC * D * 2;   // one [64][D] bf16 tile
    static constexpr int q = 0;
    static constexpr int k0 = q + kTile, v0 = k0 + kTile, k1 = v0 + kTile, v1 = k1 + kTile;   // two stages
    static constexpr int kst = v1 + kTile;                  // bf16 [S][D]: K~ at the chunk start
    static constexpr int vst = kst + S * D * 2;             // bf16 [S][D]: V~ at the chunk start
    static constexpr int wend = vst + S * D * 2;            // bf16 [S][64]: Wend
    static constexpr int beta = wend + S * 128;             // bf16 [S][64]: beta_j(u)
    static constexpr int pa = beta + S * 128;               // bf16 [64][64]: p o A (columns >= S zero)
    static constexpr int gm = pa + kDC * 128;               // bf16 [64][64]: G (upper triangle zero)
    static constexpr int pf = gm + kDC * 128;               // fp32 [64][kFS]: P; then bf16 [64][D]: O
    static constexpr int yf = pf + kDC * kFS * 4;           // fp32 [64][kFS]: Y, s, then p
    static constexpr int df = yf + kDC * kFS * 4;           // fp32 [64][kFS]: D_j(t0 + u)
    static constexpr int af = df + kDC * kFS * 4;           // fp32 [64][kFS]: alpha_j(tau)
    static constexpr int g4 = af + kDC * kFS * 4;           // fp32 [4][S]: sub-block products g_j(B)
    static constexpr int gpre = g4 + 4 * S * 4;             // fp32 [4][S]: prod_{B' < B} g_j(B')
    static constexpr int aend = gpre + 4 * S * 4;           // fp32 [S]: A_j(63)
    static constexpr int delta = aend + S * 4;              // int [S]
    static constexpr int tot = delta + S * 4;               // fp32 [kDThreads / S][S]: segment products
    static constexpr int bars = tot + kDThreads * 4;        // 3 mbarriers (q, kv stage 0, kv stage 1)
    static constexpr int total = bars + 64;
    static_assert(pf % 1024 == 0 && kst % 1024 == 0 && wend % 1024 == 0 && beta % 1024 == 0 && pa % 1024 == 0 &&
                      gm % 1024 == 0,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(total <= 227 * 1024, "shared memory of one CTA");
    static_assert(kDC * D * 2 <= kDC * kFS * 4, "the O tile reuses the P tile");
};

struct DcArgs {
    int L, G, cps, H, mode;     // mode 0: segment deltas (G > 1); 1: outputs
    long long pos0;
    float scale;
    int dmax;
    const float *Dx;            // D_M table: D_j(pos0 + t) = Dx[t + dmax - Delta_j]
    const int *delta;           // [S] slot lags
    int hs_dx, hs_delta;        // per-head strides (0: one shared period)
    const float *state_in;      // [BH][2][S][D] or null (zero state)
    float *state_out;           // [BH][2][S][D] or null
    float *seg_delta;           // [BH][G][2][S][D]: mode 0 output (state delta of each segment)
    float *seg_decay;           // [BH][G][S]: mode 0 output (prod of a_j over each segment)
    const float *win;           // [BH][G][2][S][D]: state entering each segment (G > 1)
    float *lse;                 // [BH][L]
    int *err;
};

template <int D, int S>
__global__ void __launch_bounds__(kDThreads, 1)
    k_dchunk(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
             const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o, DcArgs a) {
    using Lay = DcLayout<D, S>;
    constexpr int SPT = S / 16;                  // slots per thread in the triangle sums
    constexpr int NU = S * D / 2048;             // 16x16 state blocks per warp (K and V together)
    constexpr int SB = S / 16, DB = D / 16;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (16 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int G = a.G;
    const int bh = blockIdx.x / G, seg = blockIdx.x % G;
    if (a.mode == 0 && seg == G - 1) return;      // the last segment's delta is never used
    const int hd = bh % a.H;
    const float *Dx = a.Dx + (size_t)hd * a.hs_dx;
    const int c_begin = seg * a.cps;
    const int nch = (a.L + kDC - 1) / kDC;
    const int c_end = min(nch, c_begin + a.cps);
    const bool outputs = a.mode == 1;

    uint8_t *sQ = dsm + Lay::q, *sKst = dsm + Lay::kst, *sVst = dsm + Lay::vst, *sW = dsm + Lay::wend;
    uint8_t *sBeta = dsm + Lay::beta;
    uint8_t *sPA = dsm + Lay::pa, *sGm = dsm + Lay::gm, *sO = dsm + Lay::pf;
    float *sP = reinterpret_cast<float *>(dsm + Lay::pf), *sY = reinterpret_cast<float *>(dsm + Lay::yf);
    float *sD = reinterpret_cast<float *>(dsm + Lay::df), *sAl = reinterpret_cast<float *>(dsm + Lay::af);
    float *sG4 = reinterpret_cast<float *>(dsm + Lay::g4), *sGpre = reinterpret_cast<float *>(dsm + Lay::gpre);
    float *sAend = reinterpret_cast<float *>(dsm + Lay::aend);
    int *sdelta = reinterpret_cast<int *>(dsm + Lay::delta);
    float *sTot = reinterpret_cast<float *>(dsm + Lay::tot);
    uint64_t *bar = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    const uint32_t uQ = tc::smem_u32(sQ), uKst = tc::smem_u32(sKst), uVst = tc::smem_u32(sVst);
    const uint32_t uW = tc::smem_u32(sW), uPA = tc::smem_u32(sPA), uGm = tc::smem_u32(sGm);
    const uint32_t uBeta = tc::smem_u32(sBeta);

    if (threadIdx.x == 0) {
        for (int i = 0; i < 3; ++i) tc::mbar_init(&bar[i], 1);
        tc::fence_barrier_init();
    }
    for (int j = threadIdx.x; j < S; j += kDThreads) sdelta[j] = a.delta[(size_t)hd * a.hs_delta + j];
    // G's upper triangle and p o A's columns past S stay zero for the whole call
    for (int i = threadIdx.x; i < kDC * 64 / 2; i += kDThreads) {
        reinterpret_cast<uint32_t *>(sGm)[i] = 0u;
        reinterpret_cast<uint32_t *>(sPA)[i] = 0u;
    }
    __syncthreads();

    // ---- the state, in the accumulator layout of the state-update MMA: warp w holds NU blocks of
    // 16 rows (slots) x 16 columns of [K~ | V~]; block b -> kv = b / (SB DB), slot block, column block
    float st[NU][2][4];
    // outputs: the state entering the segment (from the scan, or the call's initial state when the
    // head is one segment); segment deltas: the zero state
    const float *src = nullptr;
    if (outputs && G > 1) src = a.win + ((size_t)bh * G + seg) * 2 * S * D;
    else if (outputs && a.state_in) src = a.state_in + (size_t)bh * 2 * S * D;
    const int g8 = lane >> 2, t4 = lane & 3;
#pragma unroll
    for (int i = 0; i < NU; ++i) {
        const int b = warp * NU + i, kv = b / (SB * DB), rem = b % (SB * DB);
        const int j0 = (rem / DB) * 16, e0 = (rem % DB) * 16;
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = j0 + g8 + ((q >> 1) << 3), e = e0 + h * 8 + 2 * t4 + (q & 1);
                st[i][h][q] = src ? src[((size_t)kv * S + j) * D + e] : 0.f;
            }
    }
    // bf16 copy of the entering state for the first chunk's Y and O
    auto store_state_copy = [&]() {
#pragma unroll
        for (int i = 0; i < NU; ++i) {
            const int b = warp * NU + i, kv = b / (SB * DB), rem = b % (SB * DB);
            const int j0 = (rem / DB) * 16, e0 = (rem % DB) * 16;
            uint8_t *tile = kv ? sVst : sKst;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int e = e0 + h * 8 + 2 * t4;
                st_bf16x2(tile, S, j0 + g8, e, st[i][h][0], st[i][h][1]);
                st_bf16x2(tile, S, j0 + g8 + 8, e, st[i][h][2], st[i][h][3]);
            }
        }
    };
    if (outputs) store_state_copy();

    // ---- TMA: q of the chunk (one buffer), k and v in two stages
    uint32_t ph_q = 0, ph_kv[2] = {0, 0};
    auto issue_q = [&](int c) {
        tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)Lay::kTile);
        for (int db = 0; db < D / 64; ++db) tc::tma_load_3d(sQ + db * kDC * 128, &tm_q, &bar[0], db * 64, c * kDC, bh);
    };
    auto issue_kv = [&](int c) {
        const int s = (c - c_begin) & 1;
        uint8_t *kb = dsm + (s ? Lay::k1 : Lay::k0), *vb = dsm + (s ? Lay::v1 : Lay::v0);
        tc::mbar_arrive_expect_tx(&bar[1 + s], (uint32_t)(2 * Lay::kTile));
        for (int db = 0; db < D / 64; ++db) {
            tc::tma_load_3d(kb + db * kDC * 128, &tm_k, &bar[1 + s], db * 64, c * kDC, bh);
            tc::tma_load_3d(vb + db * kDC * 128, &tm_v, &bar[1 + s], db * 64, c * kDC, bh);
        }
    };
    if (threadIdx.x == 0 && c_begin < c_end) {
        if (outputs) issue_q(c_begin);
        issue_kv(c_begin);
        if (c_begin + 1 < c_end) issue_kv(c_begin + 1);
    }
    float seg_dec = 1.f;   // mode 0: prod of a_j over the segment (thread j < S)
    bool ok = true;
    // ---- the decay tables of a chunk, by all threads: thread (slot j, run r) holds UPS consecutive
    // tokens' D_j; their values for the next chunk are loaded while this chunk is processed
    constexpr int NRUN = kDThreads / S, UPS = kDC / NRUN;
    const int tj = threadIdx.x % S, trun = threadIdx.x / S, tu0 = trun * UPS;
    float dl[UPS];
    auto load_d = [&](int c) {
        const int t0 = c * kDC, n = min(kDC, a.L - t0);
        const float *src = Dx + t0 + tu0 + a.dmax - sdelta[tj];
#pragma unroll
        for (int i = 0; i < UPS; ++i) dl[i] = (tu0 + i < n) ? src[i] : 0.f;
    };
    if (c_begin < c_end) load_d(c_begin);

    for (int c = c_begin; c < c_end && ok; ++c) {
        const int t0 = c * kDC, n = min(kDC, a.L - t0), s = (c - c_begin) & 1;
        const uint8_t *sK = dsm + (s ? Lay::k1 : Lay::k0), *sV = dsm + (s ? Lay::v1 : Lay::v0);
        const uint32_t uK = tc::smem_u32(sK), uV = tc::smem_u32(sV);
        // ---- D_j(t0 + u) (0 past the end of the sequence: those steps leave the state as it is) and the
        // products built from a_j = 1 - D_j, per 16-token sub-block B of the chunk:
        //   alpha_j(tau) = prod_{B start <= x <= tau} a_j,   beta_j(u) = D_j(u) prod_{u < x <= B end} a_j,
        //   g_j(B) = prod_{x in B} a_j,   Gpre_j(B) = prod_{B' < B} g_j(B')   (A_j(tau) = Gpre_j alpha_j),
        //   Wend[j][u] = D_j(u) prod_{x > u} a_j.
        // Each thread's run of UPS tokens forms its local products; the runs' totals combine through
        // shared memory.
        {
            float pf[UPS], tot = 1.f;
#pragma unroll
            for (int i = 0; i < UPS; ++i) {
                sD[(tu0 + i) * kFS + tj] = dl[i];
                tot *= 1.f - dl[i];
                pf[i] = tot;
            }
            sTot[trun * S + tj] = tot;
            if (threadIdx.x == 0) tc::bulk_wait_read0();   // the last chunk's o has left the P tile
            __syncthreads();
            constexpr int RPB = 16 / UPS;   // runs per sub-block
            const int rb0 = (trun / RPB) * RPB;
            float pre = 1.f, suf = 1.f, pre_b = 1.f, suf_b = 1.f;
            for (int r2 = 0; r2 < NRUN; ++r2) {
                const float x = sTot[r2 * S + tj];
                if (r2 < trun) {
                    pre *= x;
                    if (r2 >= rb0) pre_b *= x;
                } else if (r2 > trun) {
                    suf *= x;
                    if (r2 < rb0 + RPB) suf_b *= x;
                }
            }
#pragma unroll
            for (int i = 0; i < UPS; ++i) sAl[(tu0 + i) * kFS + tj] = pre_b * pf[i];
            if (trun == rb0) {
                // this sub-block's product and the product of the sub-blocks before it
                float gb = tot;
                for (int r2 = trun + 1; r2 < rb0 + RPB; ++r2) gb *= sTot[r2 * S + tj];
                sG4[(trun / RPB) * S + tj] = gb;
                sGpre[(trun / RPB) * S + tj] = pre;
            }
            if (trun == NRUN - 1) {
                sAend[tj] = pre * tot;
                seg_dec *= pre * tot;
            }
            float r = 1.f;   // prod of a over this run's tokens after the current one
#pragma unroll
            for (int i = UPS - 1; i >= 1; i -= 2) {
                const float w1 = dl[i] * r;
                r -= r * dl[i];
                const float w0 = dl[i - 1] * r;
                r -= r * dl[i - 1];
                st_bf16x2(sW, S, tj, tu0 + i - 1, w0 * suf, w1 * suf);
                st_bf16x2(sBeta, S, tj, tu0 + i - 1, w0 * suf_b, w1 * suf_b);
            }
        }
        if (c + 1 < c_end) load_d(c + 1);
        if (outputs) {
            // ---- P = Q K^T and Y = Q K~^T: one 16x16 block of each per warp
            if (!tc::mbar_wait(&bar[0], ph_q)) { report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (16 << 4)); ok = false; }
            ph_q ^= 1;
            if (!tc::mbar_wait(&bar[1 + s], ph_kv[s] & 1)) { report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (16 << 4)); ok = false; }
            if (!ok) break;
            // warp (sub-block bt, 16 columns): P's block, and Y's block where the columns are slots; the
            // two share Q's fragments.  Y = Q K~^T stays in registers until P is complete.
            const int bt = warp >> 2, yn0 = (warp & 3) * 16, ym0 = bt * 16;
            const bool has_y = (warp & 3) < SB;
            float yacc[2][4] = {};
            {
                float acc[2][4] = {};
                for (int k0 = 0; k0 < D; k0 += 16) {
                    uint32_t af[4], b[4];
                    load_a(uQ, kDC, ym0, k0, af);
                    load_b_nk(uK, kDC, yn0, k0, b);
                    mma16816(acc[0], af, b[0], b[1]);
                    mma16816(acc[1], af, b[2], b[3]);
                    if (has_y) {
                        load_b_nk(uKst, S, yn0, k0, b);
                        mma16816(yacc[0], af, b[0], b[1]);
                        mma16816(yacc[1], af, b[2], b[3]);
                    }
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int col = yn0 + h * 8 + 2 * t4;
                    *reinterpret_cast<float2 *>(&sP[(ym0 + g8) * kFS + col]) = make_float2(acc[h][0], acc[h][1]);
                    *reinterpret_cast<float2 *>(&sP[(ym0 + g8 + 8) * kFS + col]) = make_float2(acc[h][2], acc[h][3]);
                }
            }
            __syncthreads();
            // the next chunk's q may load now (its tile has been read)
            if (threadIdx.x == 0 && c + 1 < c_end) issue_q(c + 1);
            // ---- s[tau, j] = scale (A_j(tau) Y[tau, j] + sum_{u <= tau} P[tau, u] W_j(tau, u)).  For u in a
            // sub-block B_u before tau's, W = alpha_j(tau) gamma_j beta_j(u), gamma_j the product of g_j over
            // the sub-blocks between, so those terms are alpha_j(tau) F with
            //   F = sum_{B_u < B_tau} gamma_j P_blk beta_blk   (Horner over B_u: F <- g_j(B_u) F + P_blk beta_blk)
            // on the tensor cores; with A = Gpre alpha the warp leaves alpha (Gpre Y + F) in sY.
            if (has_y) {
                float facc[2][4] = {};
                for (int kb = 0; kb < bt; ++kb) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const float2 gk = *reinterpret_cast<const float2 *>(&sG4[kb * S + yn0 + h * 8 + 2 * t4]);
                        facc[h][0] *= gk.x; facc[h][1] *= gk.y; facc[h][2] *= gk.x; facc[h][3] *= gk.y;
                    }
                    const float *p0 = sP + (ym0 + g8) * kFS + kb * 16 + 2 * t4, *p1 = p0 + 8 * kFS;
                    const uint32_t af[4] = {tc::pack_bf16x2(p0[0], p0[1]), tc::pack_bf16x2(p1[0], p1[1]),
                                            tc::pack_bf16x2(p0[8], p0[9]), tc::pack_bf16x2(p1[8], p1[9])};
                    uint32_t b[4];
                    load_b_nk(uBeta, S, yn0, kb * 16, b);
                    mma16816(facc[0], af, b[0], b[1]);
                    mma16816(facc[1], af, b[2], b[3]);
                }
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int row = ym0 + g8 + ((q >> 1) << 3), j = yn0 + h * 8 + 2 * t4 + (q & 1);
                        sY[row * kFS + j] = sAl[row * kFS + j] * fmaf(sGpre[bt * S + j], yacc[h][q], facc[h][q]);
                    }
            }
            __syncthreads();
            // ---- the diagonal sub-blocks on the CUDA cores: thread (pair ip of sub-block sb, slot group sg)
            // walks rows 16 sb + ip and 16 sb + 15 - ip (17 steps together) down to the sub-block's start,
            // with the running product r_j
            const int sg = threadIdx.x & 15, rp = threadIdx.x >> 4, sb = rp >> 3, ip = rp & 7;
#pragma unroll 1
            for (int rr = 0; rr < 2; ++rr) {
                const int row = sb * 16 + (rr ? 15 - ip : ip), lo = sb * 16;
                float acc[SPT], r[SPT];
#pragma unroll
                for (int k = 0; k < SPT; ++k) { acc[k] = 0.f; r[k] = 1.f; }
                const float *prow = sP + row * kFS;
#pragma unroll 4
                for (int u = row; u >= lo; --u) {
                    const float pv = prow[u];
                    float dv[SPT];
                    if constexpr (SPT == 4) {
                        const float4 d4 = *reinterpret_cast<const float4 *>(&sD[u * kFS + sg * 4]);
                        dv[0] = d4.x; dv[1] = d4.y; dv[2] = d4.z; dv[3] = d4.w;
                    } else {
                        const float2 d2 = *reinterpret_cast<const float2 *>(&sD[u * kFS + sg * 2]);
                        dv[0] = d2.x; dv[1] = d2.y;
                    }
#pragma unroll
                    for (int k = 0; k < SPT; ++k) {
                        acc[k] = fmaf(pv, dv[k] * r[k], acc[k]);
                        r[k] = fmaf(-r[k], dv[k], r[k]);
                    }
                }
                const long long t = a.pos0 + t0 + row;
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    const int j = sg * SPT + k;
                    const float sc = a.scale * (sY[row * kFS + j] + acc[k]);
                    sY[row * kFS + j] = (t >= sdelta[j]) ? sc : -INFINITY;
                }
            }
            __syncthreads();
            // ---- softmax over the slots: eight threads per row
            {
                constexpr int SPR = S / 8;
                const int row = threadIdx.x >> 3, sub = threadIdx.x & 7;
                float v[SPR], mx = -INFINITY;
#pragma unroll
                for (int k = 0; k < SPR; ++k) {
                    v[k] = sY[row * kFS + sub * SPR + k];
                    mx = fmaxf(mx, v[k]);
                }
#pragma unroll
                for (int o = 4; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
                float sum = 0.f;
#pragma unroll
                for (int k = 0; k < SPR; ++k) {
                    v[k] = __expf(v[k] - mx);
                    sum += v[k];
                }
#pragma unroll
                for (int o = 4; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
                const float inv = 1.f / sum;
#pragma unroll
                for (int k = 0; k < SPR; k += 2) {
                    const int j = sub * SPR + k;
                    const float p0 = v[k] * inv, p1 = v[k + 1] * inv;
                    sY[row * kFS + j] = p0;
                    sY[row * kFS + j + 1] = p1;
                    const float g0 = sGpre[(row >> 4) * S + j], g1 = sGpre[(row >> 4) * S + j + 1];
                    st_bf16x2(sPA, kDC, row, j, p0 * g0 * sAl[row * kFS + j], p1 * g1 * sAl[row * kFS + j + 1]);
                }
                if (sub == 0 && row < n) a.lse[(size_t)bh * a.L + t0 + row] = mx + __logf(sum);
            }
            __syncthreads();
            // ---- G[tau, u] = sum_j p[tau, j] W_j(tau, u).  Diagonal sub-blocks on the CUDA cores: the walk
            // above with q_j = p_j r_j, the 16 slot groups of a row adding their partial sums by shuffles
            // within their half-warp (the two half-warps of a warp walk rows of different lengths).
            const unsigned hmask = 0xffffu << (lane & 16);
#pragma unroll 1
            for (int rr = 0; rr < 2; ++rr) {
                const int row = sb * 16 + (rr ? 15 - ip : ip), span = row - sb * 16;   // u = row - i, i <= span
                float qv[SPT], gp[16];
#pragma unroll
                for (int k = 0; k < SPT; ++k) qv[k] = sY[row * kFS + sg * SPT + k];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    gp[i] = 0.f;
                    if (i <= span) {
                        const int u = row - i;
                        float dv[SPT];
                        if constexpr (SPT == 4) {
                            const float4 d4 = *reinterpret_cast<const float4 *>(&sD[u * kFS + sg * 4]);
                            dv[0] = d4.x; dv[1] = d4.y; dv[2] = d4.z; dv[3] = d4.w;
                        } else {
                            const float2 d2 = *reinterpret_cast<const float2 *>(&sD[u * kFS + sg * 2]);
                            dv[0] = d2.x; dv[1] = d2.y;
                        }
#pragma unroll
                        for (int k = 0; k < SPT; ++k) {
                            gp[i] = fmaf(qv[k], dv[k], gp[i]);
                            qv[k] = fmaf(-qv[k], dv[k], qv[k]);
                        }
                    }
                }
                // transposing butterfly over the 16 slot groups: after the stage of width o a lane with bit
                // o set holds in gp[i] the sums of entries i + o; at the end lane sg holds entry sg
#pragma unroll
                for (int o = 8; o >= 1; o >>= 1) {
                    const bool up = (sg & o) != 0;
#pragma unroll
                    for (int i = 0; i < o; ++i) {
                        const float send = up ? gp[i] : gp[i + o];
                        const float mine = up ? gp[i + o] : gp[i];
                        gp[i] = mine + __shfl_xor_sync(hmask, send, o);
                    }
                }
                if (sg <= span)
                    *reinterpret_cast<__nv_bfloat16 *>(sGm + sw_off(kDC, row, row - sg)) = __float2bfloat16_rn(gp[0]);
            }
            // sub-blocks B_u < B_tau on the tensor cores: G_blk = (p o alpha o gamma) beta_blk^T, the
            // contraction running over the slots; warp w < 6 takes the pair (bt, bu) of w
            if (warp < 6) {
                const int gbt = 1 + (warp >= 1) + (warp >= 3), gbu = warp - gbt * (gbt - 1) / 2, m0 = gbt * 16;
                float acc[2][4] = {};
#pragma unroll
                for (int kk = 0; kk < S / 16; ++kk) {
                    float x[2][2][2];   // [row g8 / g8 + 8][column half][pair]
#pragma unroll
                    for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int j = kk * 16 + ch * 8 + 2 * t4 + e;
                            float gam = 1.f;
                            for (int b2 = gbu + 1; b2 < gbt; ++b2) gam *= sG4[b2 * S + j];
#pragma unroll
                            for (int rh = 0; rh < 2; ++rh) {
                                const int row = m0 + g8 + rh * 8;
                                x[rh][ch][e] = sY[row * kFS + j] * sAl[row * kFS + j] * gam;
                            }
                        }
                    const uint32_t af[4] = {tc::pack_bf16x2(x[0][0][0], x[0][0][1]), tc::pack_bf16x2(x[1][0][0], x[1][0][1]),
                                            tc::pack_bf16x2(x[0][1][0], x[0][1][1]), tc::pack_bf16x2(x[1][1][0], x[1][1][1])};
                    uint32_t b[4];
                    load_b_kn(uBeta, S, gbu * 16, kk * 16, b);
                    mma16816(acc[0], af, b[0], b[1]);
                    mma16816(acc[1], af, b[2], b[3]);
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int col = gbu * 16 + h * 8 + 2 * t4;
                    st_bf16x2(sGm, kDC, m0 + g8, col, acc[h][0], acc[h][1]);
                    st_bf16x2(sGm, kDC, m0 + g8 + 8, col, acc[h][2], acc[h][3]);
                }
            }
            __syncthreads();
            // ---- O = (p o A) V~ + G V_c into the O tile (over the dead P tile)
            {
                constexpr int ONB = D / 64;                      // 16-column blocks per warp
                const int m0 = (warp >> 2) * 16, nb0 = (warp & 3) * ONB * 16;
                float acc[ONB][2][4] = {};
                for (int k0 = 0; k0 < S; k0 += 16) {
                    uint32_t af[4], b[4];
                    load_a(uPA, kDC, m0, k0, af);
#pragma unroll
                    for (int nb = 0; nb < ONB; ++nb) {
                        load_b_kn(uVst, S, nb0 + nb * 16, k0, b);
                        mma16816(acc[nb][0], af, b[0], b[1]);
                        mma16816(acc[nb][1], af, b[2], b[3]);
                    }
                }
                for (int k0 = 0; k0 < kDC; k0 += 16) {
                    uint32_t af[4], b[4];
                    load_a(uGm, kDC, m0, k0, af);
#pragma unroll
                    for (int nb = 0; nb < ONB; ++nb) {
                        load_b_kn(uV, kDC, nb0 + nb * 16, k0, b);
                        mma16816(acc[nb][0], af, b[0], b[1]);
                        mma16816(acc[nb][1], af, b[2], b[3]);
                    }
                }
#pragma unroll
                for (int nb = 0; nb < ONB; ++nb)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int col = nb0 + nb * 16 + h * 8 + 2 * t4;
                        st_bf16x2(sO, kDC, m0 + g8, col, acc[nb][h][0], acc[nb][h][1]);
                        st_bf16x2(sO, kDC, m0 + g8 + 8, col, acc[nb][h][2], acc[nb][h][3]);
                    }
            }
        } else {
            if (!tc::mbar_wait(&bar[1 + s], ph_kv[s] & 1)) {
                report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (16 << 4));
                ok = false;
                break;
            }
            __syncthreads();   // A_end and Wend of this chunk
        }
        ph_kv[s] ^= 1;
        // ---- state update: X~ <- A_end o X~ + Wend X_c (every warp: its NU state blocks, which share
        // their slot rows and so Wend's fragments)
        {
            const int b0 = warp * NU, kv = b0 / (SB * DB), rem0 = b0 % (SB * DB);
            const int j0 = (rem0 / DB) * 16, e00 = (rem0 % DB) * 16;
            const float f0 = sAend[j0 + g8], f1 = sAend[j0 + g8 + 8];
#pragma unroll
            for (int i = 0; i < NU; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    st[i][h][0] *= f0; st[i][h][1] *= f0;
                    st[i][h][2] *= f1; st[i][h][3] *= f1;
                }
            const uint32_t ux = kv ? uV : uK;
            for (int k0 = 0; k0 < kDC; k0 += 16) {
                uint32_t af[4], b[4];
                load_a(uW, S, j0, k0, af);
#pragma unroll
                for (int i = 0; i < NU; ++i) {
                    load_b_kn(ux, kDC, e00 + i * 16, k0, b);
                    mma16816(st[i][0], af, b[0], b[1]);
                    mma16816(st[i][1], af, b[2], b[3]);
                }
            }
        }
        __syncthreads();   // Y and O have read the old state copy; every warp is done with this stage
        if (threadIdx.x == 0 && c + 2 < c_end) issue_kv(c + 2);
        if (outputs) {
            store_state_copy();
            // o of the chunk: one bulk tensor store (rows past the end of the sequence are clipped)
            tc::fence_proxy_async_smem();
            __syncthreads();
            if (threadIdx.x == 0) {
                for (int db = 0; db < D / 64; ++db) tc::tma_store_3d(&tm_o, sO + db * kDC * 128, db * 64, t0, bh);
                tc::bulk_commit();   // the store's read of the O tile is awaited before P is written over it
            }
        }
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
    if (!ok) return;
    // ---- results: the final state (last segment) or the segment's delta and decay product
    float *dst = nullptr;
    if (a.mode == 0) {
        dst = a.seg_delta + ((size_t)bh * G + seg) * 2 * S * D;
        if (trun == NRUN - 1) a.seg_decay[((size_t)bh * G + seg) * S + tj] = seg_dec;
    } else if (seg == G - 1 && a.state_out) {
        dst = a.state_out + (size_t)bh * 2 * S * D;
    }
    if (dst) {
#pragma unroll
        for (int i = 0; i < NU; ++i) {
            const int b = warp * NU + i, kv = b / (SB * DB), rem = b % (SB * DB);
            const int j0 = (rem / DB) * 16, e0 = (rem % DB) * 16;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int e = e0 + h * 8 + 2 * t4;
                *reinterpret_cast<float2 *>(&dst[((size_t)kv * S + j0 + g8) * D + e]) = make_float2(st[i][h][0], st[i][h][1]);
                *reinterpret_cast<float2 *>(&dst[((size_t)kv * S + j0 + g8 + 8) * D + e]) =
                    make_float2(st[i][h][2], st[i][h][3]);
            }
        }
    }
}

// States entering each segment: X_in(0) = the call's initial state (or zero);
// X_in(g+1) = prod_{segment g} a_j o X_in(g) + delta(g).  One thread per (head, K|V, slot, column).
__global__ void k_dchunk_scan(int G, int S, int D, long long total, const float *__restrict__ state_in,
                              const float *__restrict__ seg_delta, const float *__restrict__ seg_decay,
                              float *__restrict__ win) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const long long sd = (long long)S * D;
        const long long r = i / sd, within = i % sd;   // r = bh * 2 + kv
        const long long bh = r / 2, kv = r % 2;
        const int j = (int)(within / D);
        float x = state_in ? state_in[i] : 0.f;
        for (int g = 0; g < G; ++g) {
            const size_t base = ((size_t)(bh * G + g) * 2 + kv) * sd + within;
            win[base] = x;
            if (g + 1 < G) x = fmaf(seg_decay[(size_t)(bh * G + g) * S + j], x, seg_delta[base]);
        }
    }
}

template <int D, int S>
cudaError_t launch_dchunk_t(const OpDims &d, const DcArgs &base, const DcPlan &pl, const void *q, const void *k,
                            const void *v, void *o, cudaStream_t st) {
    CUtensorMap tq, tk, tv, to;
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d.L, (uint64_t)d.B * d.H};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d.L * D * 2};
    const uint32_t box[3] = {64, (uint32_t)kDC, 1};
    if (!make_tmap_bf16(&tq, q, 3, dims, strides, box) || !make_tmap_bf16(&tk, k, 3, dims, strides, box) ||
        !make_tmap_bf16(&tv, v, 3, dims, strides, box) || !make_tmap_bf16(&to, o, 3, dims, strides, box))
        return cudaErrorInvalidValue;
    const int smem = DcLayout<D, S>::total;
    cudaError_t e = cudaFuncSetAttribute(k_dchunk<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const unsigned blocks = (unsigned)((long long)d.B * d.H * pl.G);
    DcArgs a = base;
    if (pl.G > 1) {
        a.mode = 0;
        {
            ProfScope ps(BLA_K_DECAY, st);
            k_dchunk<D, S><<<blocks, kDThreads, smem, st>>>(tq, tk, tv, to, a);
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        const long long total = (long long)d.B * d.H * 2 * S * D;
        const int sblocks = (int)((total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096);
        {
            ProfScope ps(BLA_K_DECAY, st);
            k_dchunk_scan<<<sblocks, 256, 0, st>>>(pl.G, S, D, total, a.state_in, a.seg_delta, a.seg_decay,
                                                  const_cast<float *>(a.win));
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    a.mode = 1;
    ProfScope ps(BLA_K_DECAY, st);
    k_dchunk<D, S><<<blocks, kDThreads, smem, st>>>(tq, tk, tv, to, a);
    return cudaGetLastError();
}

int sm_count_dc() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 152;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 152;
    return n;
}

}  // namespace

bool decay_chunk_supported(const OpDims &d) {
    return d.dtype == BLA_BF16 && d.dk == d.dv && (d.dk == 64 || d.dk == 128) && (d.S == 32 || d.S == 64) &&
           d.L > 0;
}

// Segments per head: one CTA per SM and per segment, as many segments as fill the SMs once.
DcPlan decay_chunk_plan(const OpDims &d) {
    DcPlan p;
    const int nch = (d.L + kDC - 1) / kDC;
    const long long BH = (long long)d.B * d.H;
    long long G = sm_count_dc() / (BH > 0 ? BH : 1);
    if (G < 1) G = 1;
    if (G > nch) G = nch;
    p.cps = (int)((nch + G - 1) / G);
    p.G = (nch + p.cps - 1) / p.cps;
    return p;
}

cudaError_t launch_decay_chunk(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                               int hs_dx, int hs_delta, const void *q, const void *k, const void *v, void *o,
                               float *lse, const float *state_in, float *state_out, float *seg_delta,
                               float *seg_decay, float *win, cudaStream_t st) {
    const DcPlan pl = decay_chunk_plan(d);
    DcArgs a;
    a.L = d.L; a.G = pl.G; a.cps = pl.cps; a.H = d.H; a.mode = 1;
    a.pos0 = pos0; a.scale = d.scale; a.dmax = dmax;
    a.Dx = Dx; a.delta = delta; a.hs_dx = hs_dx; a.hs_delta = hs_delta;
    a.state_in = state_in; a.state_out = state_out;
    a.seg_delta = seg_delta; a.seg_decay = seg_decay; a.win = win;
    a.lse = lse;
    a.err = device_error_word();
    if (d.dk == 64) return d.S == 32 ? launch_dchunk_t<64, 32>(d, a, pl, q, k, v, o, st)
                                     : launch_dchunk_t<64, 64>(d, a, pl, q, k, v, o, st);
    return d.S == 32 ? launch_dchunk_t<128, 32>(d, a, pl, q, k, v, o, st)
                     : launch_dchunk_t<128, 64>(d, a, pl, q, k, v, o, st);
}

}  // namespace bla
