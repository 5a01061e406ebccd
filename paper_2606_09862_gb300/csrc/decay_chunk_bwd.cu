// decay_chunk_bwd.cu -- vector-Jacobian product of the decayed forward (Sec. 3.3) in chunks of 32
// tokens, bf16 operands, fp32 accumulation.
//
// With the chunk algebra of the forward (decay_chunk.cu): the state entering chunk c is K0, V0;
// A_j(tau), W_j(tau, u) and Wend are products of a_j = 1 - D_j; P = Q K^T, Y = Q K0^T, and
//     s = scale (A o Y + sum_u P o W),  p = softmax(s),  o = (p o A) V0 + G V,  G = sum_j p W,
//     K~end = A_end o K0 + Wend K,  V~end = A_end o V0 + Wend V.
// Given dO and the adjoints mu_K, mu_V of the states at the chunk's end (zero after the last
// chunk: the final state is not differentiated), the chain rule gives, with PV = dO V^T and
// YV = dO V0^T,
//     dp = A o YV + sum_u PV o W,   delta = sum_j p dp,   g = scale p o (dp - delta),
//     G^ = sum_j g W,
//     dQ = (g o A) K0 + G^ K,   dK = G^T Q + Wend^T mu_K,   dV = G^T dO + Wend^T mu_V,
//     mu_K <- (g o A)^T Q + A_end o mu_K,   mu_V <- (p o A)^T dO + A_end o mu_V   (the previous chunk's).
// (A numpy emulation of these lines matched the oracle's decayed VJP to 1e-15.)
//
// Both recurrences are linear with a per-slot diagonal decay, so only two thin passes run along the
// sequence; everything else runs one chunk at a time, in parallel:
//   1. k_dbtab: Wend and A_end of every (head, chunk) from the D_M table (they depend on the
//      period and the positions only, not on the batch);
//   2. k_dbstate: per (head, 64-column strip of K~ or V~): K~_{c+1} = A_end(c) o K~_c + Wend(c) K_c,
//      the state entering every chunk stored in bf16;
//   3. k_dbchain: one work item per (head, chunk), over persistent CTAs: s, p, dp, g, G, G^, then dQ
//      (final), the chunk's own parts G^T Q and G^T dO of dK and dV, and its adjoint contributions
//      Z_K = (g o A)^T Q, Z_V = (p o A)^T dO (bf16);
//   4. k_dbadj: per (head, strip), from the last chunk back: dK += Wend^T mu_K (dV likewise), then
//      mu <- A_end o mu + Z.
// In the chain the triangle sums (s, dp, G, G^) are split at 16-token sub-blocks as in the forward:
// the off-diagonal block is a contraction on the tensor cores (W = alpha_j(tau) beta_j(u) across
// adjacent sub-blocks), the diagonal blocks walk u on the CUDA cores.  All contractions are
// warp-level bf16 MMAs (m16n8k16).
#include <math.h>

#include "decay.cuh"
#include "mma_sync.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace bla {

namespace {

using namespace wmma16;

constexpr int kBC = 32;          // tokens per chunk
constexpr int kBT = 256;         // threads (8 warps)
constexpr int kBFS = kBC + 4;    // fp32 row stride of [32][32] tiles
constexpr int kBSS = 64 + 4;     // fp32 row stride of [32][S] tiles (S <= 64)

template <int D, int S>
struct BwLayout {
    static constexpr int kTile = kBC * D * 2;          // one [32][D] bf16 tile
    static constexpr int q = 0, k = q + kTile, v = k + kTile, dout = v + kTile;
    static constexpr int o = dout + kTile;              // bf16 [32][D]: dK staging (dQ is staged over v)
    static constexpr int ost = o + kTile;               // bf16 [32][D]: dV staging
    static constexpr int k0 = ost + kTile;              // bf16 [S][D]: K~ entering the chunk, then Z_K
    static constexpr int v0 = k0 + S * D * 2;           // bf16 [S][D]: V~ entering the chunk, then Z_V
    static constexpr int beta = v0 + S * D * 2;         // bf16 [S][64] (u < 32 used): beta_j(u)
    static constexpr int pa = beta + S * 128;           // bf16 [32][64]: p o A
    static constexpr int ga = pa + kBC * 128;           // bf16 [32][64]: g o A
    static constexpr int gm = ga + kBC * 128;           // bf16 [32][64] (u < 32): G
    static constexpr int gh = gm + kBC * 128;           // bf16 [32][64]: G^
    static constexpr int pf = gh + kBC * 128;           // fp32 [32][kBFS]: P
    static constexpr int pvf = pf + kBC * kBFS * 4;     // fp32 [32][kBFS]: PV
    static constexpr int sf = pvf + kBC * kBFS * 4;     // fp32 [32][kBSS]: s, then p
    static constexpr int dpf = sf + kBC * kBSS * 4;     // fp32 [32][kBSS]: dp, then g
    static constexpr int df = dpf + kBC * kBSS * 4;     // fp32 [32][kBSS]: D_j(t0 + u)
    static constexpr int af = df + kBC * kBSS * 4;      // fp32 [32][kBSS]: alpha_j(tau)
    static constexpr int g4 = af + kBC * kBSS * 4;      // fp32 [2][S]: sub-block products
    static constexpr int gpre = g4 + 2 * S * 4;         // fp32 [2][S]: product of the sub-blocks before
    static constexpr int tot = gpre + 2 * S * 4;        // fp32 [kBT / S][S]: run products
    static constexpr int delta = tot + kBT * 4;         // int [S]
    static constexpr int lse = delta + S * 4;           // fp32 [32]
    static constexpr int bars = lse + kBC * 4;          // mbarrier: the item's tiles
    static constexpr int total = bars + 64;
    static_assert(k0 % 1024 == 0 && beta % 1024 == 0 && pa % 1024 == 0 && gh % 1024 == 0 &&
                      pf % 16 == 0,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(total <= 227 * 1024, "shared memory of one CTA");
};

struct DbArgs {
    int L, H, BH;
    long long pos0;
    float scale;
    int dmax;
    const float *Dx;            // D_M table: D_j(pos0 + t) = Dx[t + dmax - Delta_j]
    const int *delta;           // [S]
    int hs_dx, hs_delta;        // per-head strides (0: one shared period)
    const float *lse;           // [BH][L], from the forward
    int ntab;                   // heads with their own tables (1 when the heads share one period)
    __nv_bfloat16 *wtab;        // [ntab][nch][S][64] bf16, 128-byte swizzled (u < 32 used): Wend
    float *atab;                // [ntab][nch][S]: A_end
    __nv_bfloat16 *states;      // [BH][nch][2][S][D]: the state entering each chunk
    __nv_bfloat16 *zbuf;        // [BH][nch][2][S][D]: each chunk's adjoint contributions (g o A)^T Q, (p o A)^T dO
    int *err;
};

// the 8 warps' share of a [2][S][D] state (K~ | V~) or of its adjoint: warp w holds NB2 blocks of 16 x 16
// in row block rb and column blocks cb0 .. cb0 + NB2 - 1 of half kv = w / 4
template <int D, int S>
struct StateMap {
    static constexpr int SB = S / 16, DB = D / 16, NB2 = SB * DB / 4;
    static_assert(NB2 >= 1 && NB2 <= DB && DB % NB2 == 0, "state blocks per warp");
    __device__ static int kv(int w) { return w >> 2; }
    __device__ static int rb(int w) { return ((w & 3) * NB2) / DB; }
    __device__ static int cb0(int w) { return ((w & 3) * NB2) % DB; }
};

template <int D, int S>
__global__ void __launch_bounds__(kBT, 1)
    k_dbchain(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
              const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
              const __grid_constant__ CUtensorMap tm_st, const __grid_constant__ CUtensorMap tm_z,
              const __grid_constant__ CUtensorMap tm_dq, const __grid_constant__ CUtensorMap tm_dk,
              const __grid_constant__ CUtensorMap tm_dv, DbArgs a) {
    using Lay = BwLayout<D, S>;
    using SMap = StateMap<D, S>;
    constexpr int SPT = S / 16, NB2 = SMap::NB2, SB = S / 16, DB = D / 16;
    constexpr int NRUN = kBT / S, UPS = kBC / NRUN, RPB = 16 / UPS;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (17 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int L = a.L, nch = (L + kBC - 1) / kBC;
    const long long nitems = (long long)a.BH * nch;
    uint8_t *sQ = dsm + Lay::q, *sK = dsm + Lay::k, *sV = dsm + Lay::v, *sDO = dsm + Lay::dout, *sO = dsm + Lay::o;
    uint8_t *sOst = dsm + Lay::ost, *sK0 = dsm + Lay::k0, *sV0 = dsm + Lay::v0, *sBeta = dsm + Lay::beta;
    uint8_t *sPA = dsm + Lay::pa, *sGA = dsm + Lay::ga, *sGm = dsm + Lay::gm, *sGh = dsm + Lay::gh;
    float *sP = reinterpret_cast<float *>(dsm + Lay::pf), *sPV = reinterpret_cast<float *>(dsm + Lay::pvf);
    float *sS = reinterpret_cast<float *>(dsm + Lay::sf), *sDP = reinterpret_cast<float *>(dsm + Lay::dpf);
    float *sD = reinterpret_cast<float *>(dsm + Lay::df), *sAl = reinterpret_cast<float *>(dsm + Lay::af);
    float *sG4 = reinterpret_cast<float *>(dsm + Lay::g4), *sGpre = reinterpret_cast<float *>(dsm + Lay::gpre);
    float *sTot = reinterpret_cast<float *>(dsm + Lay::tot);
    int *sdelta = reinterpret_cast<int *>(dsm + Lay::delta);
    float *sLse = reinterpret_cast<float *>(dsm + Lay::lse);
    uint64_t *bar = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    const uint32_t uQ = tc::smem_u32(sQ), uK = tc::smem_u32(sK), uV = tc::smem_u32(sV), uDO = tc::smem_u32(sDO);
    const uint32_t uK0 = tc::smem_u32(sK0), uV0 = tc::smem_u32(sV0), uBeta = tc::smem_u32(sBeta);
    const uint32_t uPA = tc::smem_u32(sPA), uGA = tc::smem_u32(sGA), uGm = tc::smem_u32(sGm), uGh = tc::smem_u32(sGh);

    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[0], 1);
        tc::fence_barrier_init();
    }
    // the upper triangles of G and G^, and the columns past S of p o A and g o A, stay zero
    for (int i = threadIdx.x; i < kBC * 64 / 2; i += kBT) {
        reinterpret_cast<uint32_t *>(sGm)[i] = 0u;
        reinterpret_cast<uint32_t *>(sGh)[i] = 0u;
        reinterpret_cast<uint32_t *>(sPA)[i] = 0u;
        reinterpret_cast<uint32_t *>(sGA)[i] = 0u;
    }
    __syncthreads();

    // ---- the decay tables of a chunk (as in the forward): thread (slot tj, run trun) holds UPS tokens
    const int tj = threadIdx.x % S, trun = threadIdx.x / S, tu0 = trun * UPS;
    float dl[UPS];
    auto load_d = [&](long long it) {
        const int c = (int)(it / a.BH), hd = (int)(it % a.BH) % a.H;
        const int t0 = c * kBC, n = min(kBC, L - t0);
        const float *src = a.Dx + (size_t)hd * a.hs_dx + t0 + tu0 + a.dmax - a.delta[(size_t)hd * a.hs_delta + tj];
#pragma unroll
        for (int i = 0; i < UPS; ++i) dl[i] = (tu0 + i < n) ? src[i] : 0.f;
    };
    // D_j(u), alpha_j(tau), the sub-block products g and their prefixes Gpre, and beta
    auto build_tables = [&]() {
        float pf[UPS], tot = 1.f;
#pragma unroll
        for (int i = 0; i < UPS; ++i) {
            sD[(tu0 + i) * kBSS + tj] = dl[i];
            tot *= 1.f - dl[i];
            pf[i] = tot;
        }
        sTot[trun * S + tj] = tot;
        __syncthreads();
        const int rb0 = (trun / RPB) * RPB;
        float pre = 1.f, pre_b = 1.f, suf_b = 1.f;
        for (int r2 = 0; r2 < NRUN; ++r2) {
            const float x = sTot[r2 * S + tj];
            if (r2 < trun) {
                pre *= x;
                if (r2 >= rb0) pre_b *= x;
            } else if (r2 > trun && r2 < rb0 + RPB) {
                suf_b *= x;
            }
        }
#pragma unroll
        for (int i = 0; i < UPS; ++i) sAl[(tu0 + i) * kBSS + tj] = pre_b * pf[i];
        if (trun == rb0) {
            float gb = tot;
            for (int r2 = trun + 1; r2 < rb0 + RPB; ++r2) gb *= sTot[r2 * S + tj];
            sG4[(trun / RPB) * S + tj] = gb;
            sGpre[(trun / RPB) * S + tj] = pre;
        }
        float r = 1.f;
#pragma unroll
        for (int i = UPS - 1; i >= 1; i -= 2) {
            const float w1 = dl[i] * r;
            r -= r * dl[i];
            const float w0 = dl[i - 1] * r;
            r -= r * dl[i - 1];
            st_bf16x2(sBeta, S, tj, tu0 + i - 1, w0 * suf_b, w1 * suf_b);
        }
    };

    // ---- the chunk's adjoint contributions Z, in the accumulator layout of the MMAs that form them:
    // warp w holds NB2 blocks of half kv, row block rb, column blocks cb0..
    const int skv = SMap::kv(warp), sj0 = SMap::rb(warp) * 16, se0 = SMap::cb0(warp) * 16;
    float st[NB2][2][4];
    // Z = X_a^T X (A = the transposed p o A or g o A tile, B = the chunk's q or dO)
    auto z_product = [&](uint32_t ux, uint32_t uw) {
#pragma unroll
        for (int i = 0; i < NB2; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int q = 0; q < 4; ++q) st[i][h][q] = 0.f;
        for (int k0 = 0; k0 < kBC; k0 += 16) {
            uint32_t af[4], b[4];
            load_a_t(uw, kBC, sj0, k0, af);
#pragma unroll
            for (int i = 0; i < NB2; ++i) {
                load_b_kn(ux, kBC, se0 + i * 16, k0, b);
                mma16816(st[i][0], af, b[0], b[1]);
                mma16816(st[i][1], af, b[2], b[3]);
            }
        }
    };

    uint32_t ph1 = 0;
    bool ok = true;
    const int sg = threadIdx.x & 15, rp = threadIdx.x >> 4, sb = rp >> 3, ip = rp & 7;
    const unsigned hmask = 0xffffu << (lane & 16);
    if (blockIdx.x < nitems) load_d(blockIdx.x);
    for (long long it = blockIdx.x; it < nitems && ok; it += gridDim.x) {
        const int c = (int)(it / a.BH), bh = (int)(it % a.BH), hd = bh % a.H;
        const int t0 = c * kBC, n = min(kBC, L - t0);
        const long long nx = it + gridDim.x;
        if (threadIdx.x == 0) {
            tc::bulk_wait_read0();   // the previous item's stores have read their staging tiles
            tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)(4 * Lay::kTile + 2 * S * D * 2));
            const int srow = (int)((((size_t)bh * nch + c) * 2) * S);
            for (int db = 0; db < D / 64; ++db) {
                const int x = db * 64;
                tc::tma_load_3d(sQ + db * kBC * 128, &tm_q, &bar[0], x, t0, bh);
                tc::tma_load_3d(sK + db * kBC * 128, &tm_k, &bar[0], x, t0, bh);
                tc::tma_load_3d(sV + db * kBC * 128, &tm_v, &bar[0], x, t0, bh);
                tc::tma_load_3d(sDO + db * kBC * 128, &tm_do, &bar[0], x, t0, bh);
                tc::tma_load_2d(sK0 + db * S * 128, &tm_st, &bar[0], x, srow);
                tc::tma_load_2d(sV0 + db * S * 128, &tm_st, &bar[0], x, srow + S);
            }
            // the next item's tiles into L2 meanwhile
            if (nx < nitems) {
                const int cn = (int)(nx / a.BH), bn = (int)(nx % a.BH), tn = cn * kBC;
                for (int db = 0; db < D / 64; ++db) {
                    const int x = db * 64;
                    tc::tma_prefetch_3d(&tm_q, x, tn, bn);
                    tc::tma_prefetch_3d(&tm_k, x, tn, bn);
                    tc::tma_prefetch_3d(&tm_v, x, tn, bn);
                    tc::tma_prefetch_3d(&tm_do, x, tn, bn);
                }
                tc::bulk_prefetch_l2(a.states + (((size_t)bn * nch + cn) * 2) * S * D, (uint32_t)(2 * S * D * 2));
            }
        }
        // sdelta and sLse were last read before the previous item's closing barriers
        for (int j = threadIdx.x; j < S; j += kBT) sdelta[j] = a.delta[(size_t)hd * a.hs_delta + j];
        if (threadIdx.x < kBC) sLse[threadIdx.x] = threadIdx.x < n ? a.lse[(size_t)bh * L + t0 + threadIdx.x] : 0.f;
        build_tables();
        if (nx < nitems) load_d(nx);
        if (!tc::mbar_wait(&bar[0], ph1)) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (17 << 4));
            ok = false;
            break;
        }
        ph1 ^= 1;
        // ---- (a) P = Q K^T, Y = Q K0^T (warps 0-3), PV = dO V^T, YV = dO V0^T (warps 4-7): warp takes
        // row block m0 and half hh of the columns; Y / YV stay in registers
        const int side = warp >> 2, m0 = ((warp >> 1) & 1) * 16, hh = warp & 1, bt = m0 >> 4;
        constexpr int YB = SB / 2 > 0 ? SB / 2 : 1;   // 16-column blocks of Y per warp
        const int yn0 = hh * (S / 2);
        float yacc[YB][2][4] = {};
        {
            const uint32_t ua = side ? uDO : uQ, ub = side ? uV : uK, uy = side ? uV0 : uK0;
            float pacc[2][4] = {};
            for (int k0 = 0; k0 < D; k0 += 16) {
                uint32_t af[4], b[4];
                load_a(ua, kBC, m0, k0, af);
                load_b_nk(ub, kBC, hh * 16, k0, b);
                mma16816(pacc[0], af, b[0], b[1]);
                mma16816(pacc[1], af, b[2], b[3]);
#pragma unroll
                for (int i = 0; i < YB; ++i) {
                    if (yn0 + i * 16 >= S) break;
                    load_b_nk(uy, S, yn0 + i * 16, k0, b);
                    mma16816(yacc[i][0], af, b[0], b[1]);
                    mma16816(yacc[i][1], af, b[2], b[3]);
                }
            }
            float *dst = side ? sPV : sP;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int col = hh * 16 + h * 8 + 2 * t4;
                *reinterpret_cast<float2 *>(&dst[(m0 + g8) * kBFS + col]) = make_float2(pacc[h][0], pacc[h][1]);
                *reinterpret_cast<float2 *>(&dst[(m0 + g8 + 8) * kBFS + col]) = make_float2(pacc[h][2], pacc[h][3]);
            }
        }
        __syncthreads();
        // ---- (b) the off-diagonal block of sub-block 1 over sub-block 0 (W = alpha beta there), and
        // alpha (Gpre Y + F) into s (warps 0-3) or dp (warps 4-7)
        {
            const float *pm = side ? sPV : sP;
            float *dst = side ? sDP : sS;
#pragma unroll
            for (int i = 0; i < YB; ++i) {
                const int n0 = yn0 + i * 16;
                if (n0 >= S) break;
                float facc[2][4] = {};
                if (bt == 1) {
                    const float *p0 = pm + (m0 + g8) * kBFS + 2 * t4, *p1 = p0 + 8 * kBFS;
                    const uint32_t af[4] = {tc::pack_bf16x2(p0[0], p0[1]), tc::pack_bf16x2(p1[0], p1[1]),
                                            tc::pack_bf16x2(p0[8], p0[9]), tc::pack_bf16x2(p1[8], p1[9])};
                    uint32_t b[4];
                    load_b_nk(uBeta, S, n0, 0, b);
                    mma16816(facc[0], af, b[0], b[1]);
                    mma16816(facc[1], af, b[2], b[3]);
                }
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int row = m0 + g8 + ((q >> 1) << 3), j = n0 + h * 8 + 2 * t4 + (q & 1);
                        dst[row * kBSS + j] = sAl[row * kBSS + j] * fmaf(sGpre[bt * S + j], yacc[i][h][q], facc[h][q]);
                    }
            }
        }
        __syncthreads();
        // ---- (c) the diagonal sub-blocks of s and dp on the CUDA cores (one walk, the same weights),
        // then p = exp(s - lse), delta = sum_j p dp (the 16 slot groups of the row add theirs by shuffles:
        // exact for the p and dp at hand, so a row whose softmax sees one slot gets g = 0), g = scale p
        // (dp - delta), and p o A, g o A in bf16
#pragma unroll 1
        for (int rr = 0; rr < 2; ++rr) {
            const int row = sb * 16 + (rr ? 15 - ip : ip), lo = sb * 16;
            float as[SPT], ad[SPT], r[SPT];
#pragma unroll
            for (int k = 0; k < SPT; ++k) { as[k] = 0.f; ad[k] = 0.f; r[k] = 1.f; }
#pragma unroll 4
            for (int u = row; u >= lo; --u) {
                const float pv = sP[row * kBFS + u], pw = sPV[row * kBFS + u];
                float dv[SPT];
                if constexpr (SPT == 4) {
                    const float4 d4 = *reinterpret_cast<const float4 *>(&sD[u * kBSS + sg * 4]);
                    dv[0] = d4.x; dv[1] = d4.y; dv[2] = d4.z; dv[3] = d4.w;
                } else {
                    const float2 d2 = *reinterpret_cast<const float2 *>(&sD[u * kBSS + sg * 2]);
                    dv[0] = d2.x; dv[1] = d2.y;
                }
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    const float w = dv[k] * r[k];
                    as[k] = fmaf(pv, w, as[k]);
                    ad[k] = fmaf(pw, w, ad[k]);
                    r[k] = fmaf(-r[k], dv[k], r[k]);
                }
            }
            const long long t = a.pos0 + t0 + row;
            const bool live = row < n;
            const float lr = sLse[row];
            float pj[SPT], dpj[SPT], gj[SPT], pdp = 0.f;
#pragma unroll
            for (int k = 0; k < SPT; ++k) {
                const int j = sg * SPT + k;
                const float s = a.scale * (sS[row * kBSS + j] + as[k]);
                pj[k] = (live && t >= sdelta[j]) ? __expf(s - lr) : 0.f;
                dpj[k] = sDP[row * kBSS + j] + ad[k];
                pdp = fmaf(pj[k], dpj[k], pdp);
            }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) pdp += __shfl_xor_sync(hmask, pdp, o);
#pragma unroll
            for (int k = 0; k < SPT; ++k) {
                const int j = sg * SPT + k;
                gj[k] = a.scale * pj[k] * (dpj[k] - pdp);
                sS[row * kBSS + j] = pj[k];
                sDP[row * kBSS + j] = gj[k];
            }
#pragma unroll
            for (int k = 0; k < SPT; k += 2) {
                const int j = sg * SPT + k;
                const float A0 = sGpre[sb * S + j] * sAl[row * kBSS + j];
                const float A1 = sGpre[sb * S + j + 1] * sAl[row * kBSS + j + 1];
                st_bf16x2(sPA, kBC, row, j, pj[k] * A0, pj[k + 1] * A1);
                st_bf16x2(sGA, kBC, row, j, gj[k] * A0, gj[k + 1] * A1);
            }
        }
        __syncthreads();
        // ---- (d) G = sum_j p W and G^ = sum_j g W: diagonal sub-blocks by the walk (partials per step in
        // registers, one transposing butterfly over the 16 slot groups each), the block of sub-block 1
        // over sub-block 0 on the tensor cores (warp 0: G, warp 1: G^)
#pragma unroll 1
        for (int rr = 0; rr < 2; ++rr) {
            const int row = sb * 16 + (rr ? 15 - ip : ip), span = row - sb * 16;
            float qv[SPT], hv[SPT], gp[16], hp[16];
#pragma unroll
            for (int k = 0; k < SPT; ++k) {
                qv[k] = sS[row * kBSS + sg * SPT + k];
                hv[k] = sDP[row * kBSS + sg * SPT + k];
            }
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                gp[i] = 0.f;
                hp[i] = 0.f;
                if (i <= span) {
                    const int u = row - i;
                    float dv[SPT];
                    if constexpr (SPT == 4) {
                        const float4 d4 = *reinterpret_cast<const float4 *>(&sD[u * kBSS + sg * 4]);
                        dv[0] = d4.x; dv[1] = d4.y; dv[2] = d4.z; dv[3] = d4.w;
                    } else {
                        const float2 d2 = *reinterpret_cast<const float2 *>(&sD[u * kBSS + sg * 2]);
                        dv[0] = d2.x; dv[1] = d2.y;
                    }
#pragma unroll
                    for (int k = 0; k < SPT; ++k) {
                        gp[i] = fmaf(qv[k], dv[k], gp[i]);
                        hp[i] = fmaf(hv[k], dv[k], hp[i]);
                        qv[k] = fmaf(-qv[k], dv[k], qv[k]);
                        hv[k] = fmaf(-hv[k], dv[k], hv[k]);
                    }
                }
            }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                const bool up = (sg & o) != 0;
#pragma unroll
                for (int i = 0; i < o; ++i) {
                    const float s1 = up ? gp[i] : gp[i + o], m1 = up ? gp[i + o] : gp[i];
                    const float s2 = up ? hp[i] : hp[i + o], m2 = up ? hp[i + o] : hp[i];
                    gp[i] = m1 + __shfl_xor_sync(hmask, s1, o);
                    hp[i] = m2 + __shfl_xor_sync(hmask, s2, o);
                }
            }
            if (sg <= span) {
                const uint32_t off = sw_off(kBC, row, row - sg);
                *reinterpret_cast<__nv_bfloat16 *>(sGm + off) = __float2bfloat16_rn(gp[0]);
                *reinterpret_cast<__nv_bfloat16 *>(sGh + off) = __float2bfloat16_rn(hp[0]);
            }
        }
        if (warp < 2) {
            const float *src = warp ? sDP : sS;
            float acc[2][4] = {};
#pragma unroll
            for (int kk = 0; kk < SB; ++kk) {
                float x[2][2][2];
#pragma unroll
                for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                    for (int e = 0; e < 2; ++e)
#pragma unroll
                        for (int rh = 0; rh < 2; ++rh) {
                            const int row = 16 + g8 + rh * 8, j = kk * 16 + ch * 8 + 2 * t4 + e;
                            x[rh][ch][e] = src[row * kBSS + j] * sAl[row * kBSS + j];
                        }
                const uint32_t af[4] = {tc::pack_bf16x2(x[0][0][0], x[0][0][1]), tc::pack_bf16x2(x[1][0][0], x[1][0][1]),
                                        tc::pack_bf16x2(x[0][1][0], x[0][1][1]), tc::pack_bf16x2(x[1][1][0], x[1][1][1])};
                uint32_t b[4];
                load_b_kn(uBeta, S, 0, kk * 16, b);
                mma16816(acc[0], af, b[0], b[1]);
                mma16816(acc[1], af, b[2], b[3]);
            }
            uint8_t *dst = warp ? sGh : sGm;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int col = h * 8 + 2 * t4;
                st_bf16x2(dst, kBC, 16 + g8, col, acc[h][0], acc[h][1]);
                st_bf16x2(dst, kBC, 24 + g8, col, acc[h][2], acc[h][3]);
            }
        }
        __syncthreads();
        // ---- (e) dQ = (g o A) K0 + G^ K into the v tile, dK = G^T Q + Wend^T mu_K into the o tile,
        // dV = G^T dO + Wend^T mu_V into the staging tile: warp takes row block orb and OCB column blocks
        {
            constexpr int OCB = DB / 4;
            const int om0 = (warp & 1) * 16, on0 = (warp >> 1) * OCB * 16;
            auto out3 = [&](int which) {
                float acc[OCB][2][4] = {};
                uint32_t af[4], b[4];
                if (which == 0) {
                    for (int k0 = 0; k0 < S; k0 += 16) {
                        load_a(uGA, kBC, om0, k0, af);
#pragma unroll
                        for (int cb = 0; cb < OCB; ++cb) {
                            load_b_kn(uK0, S, on0 + cb * 16, k0, b);
                            mma16816(acc[cb][0], af, b[0], b[1]);
                            mma16816(acc[cb][1], af, b[2], b[3]);
                        }
                    }
                    for (int k0 = 0; k0 < kBC; k0 += 16) {
                        load_a(uGh, kBC, om0, k0, af);
#pragma unroll
                        for (int cb = 0; cb < OCB; ++cb) {
                            load_b_kn(uK, kBC, on0 + cb * 16, k0, b);
                            mma16816(acc[cb][0], af, b[0], b[1]);
                            mma16816(acc[cb][1], af, b[2], b[3]);
                        }
                    }
                } else {
                    const uint32_t ug = which == 1 ? uGh : uGm, ux = which == 1 ? uQ : uDO;
                    for (int k0 = 0; k0 < kBC; k0 += 16) {
                        load_a_t(ug, kBC, om0, k0, af);
#pragma unroll
                        for (int cb = 0; cb < OCB; ++cb) {
                            load_b_kn(ux, kBC, on0 + cb * 16, k0, b);
                            mma16816(acc[cb][0], af, b[0], b[1]);
                            mma16816(acc[cb][1], af, b[2], b[3]);
                        }
                    }
                }
                uint8_t *dst = which == 0 ? sV : which == 1 ? sO : sOst;
#pragma unroll
                for (int cb = 0; cb < OCB; ++cb)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int col = on0 + cb * 16 + h * 8 + 2 * t4;
                        st_bf16x2(dst, kBC, om0 + g8, col, acc[cb][h][0], acc[cb][h][1]);
                        st_bf16x2(dst, kBC, om0 + g8 + 8, col, acc[cb][h][2], acc[cb][h][3]);
                    }
            };
            // dQ reads K0 and K, dK reads Q, dV reads dO: none of them reads the v or o tile, which the
            // stores overwrite (V was read by PV, o by delta, before the barriers above)
            out3(0);
            out3(1);
            out3(2);
        }
        // ---- the chunk's adjoint contributions Z_K = (g o A)^T Q, Z_V = (p o A)^T dO, staged over the
        // K0 and V0 tiles once every warp has finished dQ
        z_product(skv ? uDO : uQ, skv ? uPA : uGA);
        __syncthreads();
        {
            uint8_t *tile = skv ? sV0 : sK0;
#pragma unroll
            for (int i = 0; i < NB2; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int e = se0 + i * 16 + h * 8 + 2 * t4;
                    st_bf16x2(tile, S, sj0 + g8, e, st[i][h][0], st[i][h][1]);
                    st_bf16x2(tile, S, sj0 + g8 + 8, e, st[i][h][2], st[i][h][3]);
                }
        }
        tc::fence_proxy_async_smem();
        __syncthreads();
        if (threadIdx.x == 0) {
            const int srow = (int)((((size_t)bh * nch + c) * 2) * S);
            for (int db = 0; db < D / 64; ++db) {
                tc::tma_store_3d(&tm_dq, sV + db * kBC * 128, db * 64, t0, bh);
                tc::tma_store_3d(&tm_dk, sO + db * kBC * 128, db * 64, t0, bh);
                tc::tma_store_3d(&tm_dv, sOst + db * kBC * 128, db * 64, t0, bh);
                tc::tma_store_2d(&tm_z, sK0 + db * S * 128, db * 64, srow);
                tc::tma_store_2d(&tm_z, sV0 + db * S * 128, db * 64, srow + S);
            }
            tc::bulk_commit();
        }
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
}

// ---- Wend and A_end of every (head, chunk): thread j walks the chunk's tokens from the last back.
// D_j(t0 + u) = Dx[t0 + u + dmax - Delta_j]; tokens past L contribute nothing (D = 0).
template <int S>
__global__ void __launch_bounds__(S) k_dbtab(DbArgs a) {
    const int c = blockIdx.x, h = blockIdx.y, j = threadIdx.x, nch = (a.L + kBC - 1) / kBC;
    const int t0 = c * kBC, n = min(kBC, a.L - t0);
    const float *src = a.Dx + (size_t)h * a.hs_dx + t0 + a.dmax - a.delta[(size_t)h * a.hs_delta + j];
    uint8_t *w = reinterpret_cast<uint8_t *>(a.wtab + ((size_t)h * nch + c) * S * 64);
    float r = 1.f;
#pragma unroll 4
    for (int u = kBC - 2; u >= 0; u -= 2) {
        const float d1 = (u + 1 < n) ? src[u + 1] : 0.f, d0 = (u < n) ? src[u] : 0.f;
        const float w1 = d1 * r;
        r -= r * d1;
        const float w0 = d0 * r;
        r -= r * d0;
        *reinterpret_cast<uint32_t *>(w + wmma16::sw_off(S, j, u)) = tc::pack_bf16x2(w0, w1);
    }
    for (int u = kBC; u < 64; u += 2) *reinterpret_cast<uint32_t *>(w + wmma16::sw_off(S, j, u)) = 0u;
    a.atab[((size_t)h * nch + c) * S + j] = r;
}

// ---- the two thin passes along the sequence.  One CTA per (64-column strip, K~ or V~, head) with
// 4 warps; the strip [S][64] (fp32) lives in the accumulator registers of the MMAs that update it.
constexpr int kSW = 4;           // warps
constexpr int kNS = 4;           // pipeline stages

template <int S>
struct StripMap {
    static constexpr int WR = S / 16, WC = kSW / WR, NC = 64 / WC, NB = NC / 16;
    static_assert(WR * WC == kSW && NB >= 1, "strip blocks per warp");
};

template <int S>
struct ScanLayout {
    static constexpr int kT = kBC * 128;                    // [32][64] bf16 tile
    static constexpr int kW = S * 128;                      // [S][64] bf16 tile (Wend image, state strip)
    static constexpr int stage = kW + kW + kT;              // z (reverse only) | Wend | k or dk
    static constexpr int mu = kNS * stage;                  // bf16 [S][64]: mu (reverse)
    static constexpr int out = mu + kW;                     // 2 staging tiles: [S][64] (state) or [32][64]
    static constexpr int ae = out + 2 * kW;                 // fp32 [kNS][S]: A_end of each stage
    static constexpr int bars = ae + kNS * S * 4;
    static constexpr int total = bars + 8 * kNS;
    static_assert(stage % 1024 == 0 && mu % 1024 == 0 && out % 1024 == 0, "swizzled tiles need 1024-byte alignment");
};

// REV = false: K~_{c+1} = A_end(c) o K~_c + Wend(c) K_c from the zero state; the state entering chunk c
// goes to `states` (bf16).  REV = true: from the last chunk back, dK_c += Wend(c)^T mu_c (bf16 MMA on a
// copy of mu), then mu_{c-1} = A_end(c) o mu_c + Z_c.
template <int D, int S, bool REV>
__global__ void __launch_bounds__(kSW * 32)
    k_dbscan(const __grid_constant__ CUtensorMap tm_x0, const __grid_constant__ CUtensorMap tm_x1,
             const __grid_constant__ CUtensorMap tm_st, DbArgs a) {
    using Lay = ScanLayout<S>;
    using M = StripMap<S>;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (18 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int strip = blockIdx.x, kv = blockIdx.y, bh = blockIdx.z;
    const int tab = a.ntab > 1 ? bh % a.H : 0;
    const int nch = (a.L + kBC - 1) / kBC, x = strip * 64;
    const CUtensorMap *tx = kv ? &tm_x1 : &tm_x0;   // k / v (forward) or dk / dv (reverse)
    uint64_t *full = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    uint8_t *sMu = dsm + Lay::mu, *sOut = dsm + Lay::out;
    // stage s: Z strip (reverse) at +0, Wend at +kW, the [32][64] tile at +2 kW; its A_end apart
    auto sz = [&](int s) { return dsm + s * Lay::stage; };
    auto sw = [&](int s) { return dsm + s * Lay::stage + Lay::kW; };
    auto sx = [&](int s) { return dsm + s * Lay::stage + 2 * Lay::kW; };
    auto sa = [&](int s) { return reinterpret_cast<float *>(dsm + Lay::ae + s * S * 4); };
    auto chunk_of = [&](int i) { return REV ? nch - 1 - i : i; };
    auto issue = [&](int i) {
        const int s = i % kNS, c = chunk_of(i);
        const size_t ti = (size_t)tab * nch + c;
        const uint32_t bytes = (uint32_t)(Lay::kW + Lay::kT + S * 4 + (REV ? Lay::kW : 0));
        tc::mbar_arrive_expect_tx(&full[s], bytes);
        if (REV) tc::tma_load_2d(sz(s), &tm_st, &full[s], x, (int)((((size_t)bh * nch + c) * 2 + kv) * S));
        tc::bulk_load(sw(s), a.wtab + ti * S * 64, (uint32_t)Lay::kW, &full[s]);
        tc::tma_load_3d(sx(s), tx, &full[s], x, c * kBC, bh);
        tc::bulk_load(sa(s), a.atab + ti * S, (uint32_t)(S * 4), &full[s]);
    };
    if (threadIdx.x == 0) {
        for (int s = 0; s < kNS; ++s) tc::mbar_init(&full[s], 1);
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (int i = 0; i < kNS && i < nch; ++i) issue(i);

    const int r0 = (warp % M::WR) * 16, c0 = (warp / M::WR) * M::NC;
    float acc[M::NB][2][4];
#pragma unroll
    for (int i = 0; i < M::NB; ++i)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[i][h][q] = 0.f;
    auto put = [&](uint8_t *tile) {   // acc (bf16) into a swizzled [S][64] tile
#pragma unroll
        for (int i = 0; i < M::NB; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int e = c0 + i * 16 + h * 8 + 2 * t4;
                st_bf16x2(tile, S, r0 + g8, e, acc[i][h][0], acc[i][h][1]);
                st_bf16x2(tile, S, r0 + g8 + 8, e, acc[i][h][2], acc[i][h][3]);
            }
    };
    bool ok = true;
    for (int i = 0; i < nch; ++i) {
        const int s = i % kNS, c = chunk_of(i), ob = i & 1;
        if (threadIdx.x == 0) tc::bulk_wait_read1();   // the store that used staging tile ob has read it
        if (!REV) {
            __syncthreads();
            put(sOut + ob * Lay::kW);   // the state entering chunk c
        }
        if (!tc::mbar_wait(&full[s], (uint32_t)((i / kNS) & 1))) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (18 << 4));
            ok = false;
        }
        if (__syncthreads_or(!ok)) break;
        const float *ae = sa(s);
        const float f0 = ae[r0 + g8], f1 = ae[r0 + g8 + 8];
        const uint32_t uW = tc::smem_u32(sw(s)), uX = tc::smem_u32(sx(s));
        if (!REV) {
            // acc <- A_end o acc + Wend K_c: A = Wend [S][32 tokens], B = the chunk's strip [32][64]
#pragma unroll
            for (int b = 0; b < M::NB; ++b)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    acc[b][h][0] *= f0; acc[b][h][1] *= f0;
                    acc[b][h][2] *= f1; acc[b][h][3] *= f1;
                }
#pragma unroll
            for (int k0 = 0; k0 < kBC; k0 += 16) {
                uint32_t af[4], bf[4];
                load_a(uW, S, r0, k0, af);
#pragma unroll
                for (int b = 0; b < M::NB; ++b) {
                    load_b_kn(uX, kBC, c0 + b * 16, k0, bf);
                    mma16816(acc[b][0], af, bf[0], bf[1]);
                    mma16816(acc[b][1], af, bf[2], bf[3]);
                }
            }
        } else {
            // dK_c [32][64] += Wend^T mu: warp takes token rows om0.. and 32 columns on0..
            const bool live = i > 0;   // mu is zero after the last chunk
            if (live) {
                put(sMu);
                __syncthreads();
                const int om0 = (warp & 1) * 16, on0 = (warp >> 1) * 32;
                float o[2][2][4] = {};
                const uint32_t uMu = tc::smem_u32(sMu);
#pragma unroll
                for (int k0 = 0; k0 < S; k0 += 16) {
                    uint32_t af[4], bf[4];
                    load_a_t(uW, S, om0, k0, af);
#pragma unroll
                    for (int b = 0; b < 2; ++b) {
                        load_b_kn(uMu, S, on0 + b * 16, k0, bf);
                        mma16816(o[b][0], af, bf[0], bf[1]);
                        mma16816(o[b][1], af, bf[2], bf[3]);
                    }
                }
                const uint8_t *dk = sx(s);
                uint8_t *dst = sOut + ob * Lay::kW;
#pragma unroll
                for (int b = 0; b < 2; ++b)
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int rh = 0; rh < 2; ++rh) {
                            const int row = om0 + g8 + rh * 8, col = on0 + b * 16 + h * 8 + 2 * t4;
                            const float2 l = __bfloat1622float2(
                                *reinterpret_cast<const __nv_bfloat162 *>(dk + sw_off(kBC, row, col)));
                            st_bf16x2(dst, kBC, row, col, o[b][h][2 * rh] + l.x, o[b][h][2 * rh + 1] + l.y);
                        }
            }
            // mu <- A_end o mu + Z_c
            const uint8_t *z = sz(s);
#pragma unroll
            for (int b = 0; b < M::NB; ++b)
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int rh = 0; rh < 2; ++rh) {
                        const int row = r0 + g8 + rh * 8, col = c0 + b * 16 + h * 8 + 2 * t4;
                        const float f = rh ? f1 : f0;
                        const float2 zz =
                            __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(z + sw_off(S, row, col)));
                        acc[b][h][2 * rh] = fmaf(f, acc[b][h][2 * rh], zz.x);
                        acc[b][h][2 * rh + 1] = fmaf(f, acc[b][h][2 * rh + 1], zz.y);
                    }
        }
        tc::fence_proxy_async_smem();
        __syncthreads();   // stage s and the staging tile are complete
        if (threadIdx.x == 0) {
            if (!REV) {
                tc::tma_store_2d(&tm_st, sOut + ob * Lay::kW, x, (int)((((size_t)bh * nch + c) * 2 + kv) * S));
                tc::bulk_commit();
            } else if (i > 0) {
                tc::tma_store_3d(tx, sOut + ob * Lay::kW, x, c * kBC, bh);
                tc::bulk_commit();
            }
            if (i + kNS < nch) issue(i + kNS);
        }
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
}

int sm_count_db() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 152;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 152;
    return n;
}

template <int D, int S>
cudaError_t launch_dbwd_t(const OpDims &d, const DbArgs &a, const void *q, const void *k, const void *v,
                          const void *dout, void *dq, void *dk, void *dv, cudaStream_t st) {
    CUtensorMap tq, tk, tv, tdo, tst, tz, tdq, tdk, tdv;
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d.L, (uint64_t)d.B * d.H};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d.L * D * 2};
    const uint32_t box[3] = {64, (uint32_t)kBC, 1};
    const int nch = (d.L + kBC - 1) / kBC;
    const uint64_t sdims[2] = {(uint64_t)D, (uint64_t)d.B * d.H * nch * 2 * S};
    const uint64_t sstr[1] = {(uint64_t)D * 2};
    const uint32_t sbox[2] = {64, (uint32_t)S};
    if (!make_tmap_bf16(&tq, q, 3, dims, strides, box) || !make_tmap_bf16(&tk, k, 3, dims, strides, box) ||
        !make_tmap_bf16(&tv, v, 3, dims, strides, box) || !make_tmap_bf16(&tdo, dout, 3, dims, strides, box) ||
        !make_tmap_bf16(&tst, a.states, 2, sdims, sstr, sbox) || !make_tmap_bf16(&tz, a.zbuf, 2, sdims, sstr, sbox) ||
        !make_tmap_bf16(&tdq, dq, 3, dims, strides, box) || !make_tmap_bf16(&tdk, dk, 3, dims, strides, box) ||
        !make_tmap_bf16(&tdv, dv, 3, dims, strides, box))
        return cudaErrorInvalidValue;
    const int smem = BwLayout<D, S>::total, ssm = ScanLayout<S>::total;
    cudaError_t e = cudaFuncSetAttribute(k_dbchain<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_dbscan<D, S, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, ssm);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_dbscan<D, S, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, ssm);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_DECAY, st);
    k_dbtab<S><<<dim3((unsigned)nch, (unsigned)a.ntab), S, 0, st>>>(a);
    const dim3 sgrid((unsigned)(D / 64), 2u, (unsigned)a.BH);
    k_dbscan<D, S, false><<<sgrid, kSW * 32, ssm, st>>>(tk, tv, tst, a);
    const long long items = (long long)a.BH * nch;
    const int grid = (int)(items < sm_count_db() ? items : sm_count_db());
    k_dbchain<D, S><<<(unsigned)grid, kBT, smem, st>>>(tq, tk, tv, tdo, tst, tz, tdq, tdk, tdv, a);
    k_dbscan<D, S, true><<<sgrid, kSW * 32, ssm, st>>>(tdk, tdv, tz, a);
    return cudaGetLastError();
}

// the pieces of the backward's workspace: states, Z, Wend tables, A_end tables
struct DbWs {
    size_t states, z, wtab, atab, total;
};

DbWs db_ws(const OpDims &d) {
    const size_t nch = (size_t)(d.L + kBC - 1) / kBC, ntab = d.periods ? (size_t)d.H : 1;
    const size_t per = align_up((size_t)d.B * d.H * nch * 2 * d.S * d.dk * sizeof(__nv_bfloat16), 256);
    DbWs w;
    w.states = 0;
    w.z = per;
    w.wtab = 2 * per;
    w.atab = w.wtab + align_up(ntab * nch * d.S * 64 * sizeof(__nv_bfloat16), 256);
    w.total = w.atab + align_up(ntab * nch * d.S * sizeof(float), 256);
    return w;
}

}  // namespace

size_t decay_chunk_bwd_ws_bytes(const OpDims &d) { return db_ws(d).total; }

cudaError_t launch_decay_chunk_bwd(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                                   int hs_dx, int hs_delta, const void *q, const void *k, const void *v,
                                   const void *dout, const float *lse, void *dq, void *dk, void *dv, void *ws,
                                   cudaStream_t st) {
    const DbWs w = db_ws(d);
    char *base = static_cast<char *>(ws);
    DbArgs a;
    a.L = d.L; a.H = d.H; a.BH = d.B * d.H; a.pos0 = pos0; a.scale = d.scale; a.dmax = dmax;
    a.Dx = Dx; a.delta = delta; a.hs_dx = hs_dx; a.hs_delta = hs_delta;
    a.lse = lse;
    a.ntab = (hs_dx != 0 || hs_delta != 0) ? d.H : 1;
    if (a.ntab > 1 && !d.periods) return cudaErrorInvalidValue;   // the tables are sized per head only then
    a.states = reinterpret_cast<__nv_bfloat16 *>(base + w.states);
    a.zbuf = reinterpret_cast<__nv_bfloat16 *>(base + w.z);
    a.wtab = reinterpret_cast<__nv_bfloat16 *>(base + w.wtab);
    a.atab = reinterpret_cast<float *>(base + w.atab);
    a.err = device_error_word();
    if (d.dk == 64) return d.S == 32 ? launch_dbwd_t<64, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                                     : launch_dbwd_t<64, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
    return d.S == 32 ? launch_dbwd_t<128, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                     : launch_dbwd_t<128, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
}

}  // namespace bla
