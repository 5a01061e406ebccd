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
// One CTA per head: a forward sweep runs the state updates alone and stores the state entering
// every chunk (bf16); a reverse sweep then takes the chunks from last to first with mu in the
// accumulator registers of the MMAs that update it.  As in the forward, the triangle sums (s, dp, G,
// G^) are split at 16-token sub-blocks: the off-diagonal block is a contraction on the tensor cores
// (W = alpha_j(tau) beta_j(u) across adjacent sub-blocks), the diagonal blocks walk u on the CUDA
// cores.  All contractions are warp-level bf16 MMAs (m16n8k16).
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
    static constexpr int k0 = ost + kTile;              // bf16 [S][D]: K~ entering the chunk
    static constexpr int v0 = k0 + S * D * 2;           // bf16 [S][D]: V~ entering the chunk
    static constexpr int muk = v0 + S * D * 2;          // bf16 [S][D]: adjoint of K~ at the chunk's end
    static constexpr int muv = muk + S * D * 2;         // bf16 [S][D]: adjoint of V~
    static constexpr int wend = muv + S * D * 2;        // bf16 [S][64] (u < 32 used): Wend
    static constexpr int beta = wend + S * 128;         // bf16 [S][64]: beta_j(u)
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
    static constexpr int aend = gpre + 2 * S * 4;       // fp32 [S]
    static constexpr int tot = aend + S * 4;            // fp32 [kBT / S][S]: run products
    static constexpr int delta = tot + kBT * 4;         // int [S]
    static constexpr int lse = delta + S * 4;           // fp32 [32]
    static constexpr int bars = lse + kBC * 4;          // mbarriers: forward-sweep stages 0 and 1, reverse sweep
    static constexpr int total = bars + 64;
    static_assert(k0 % 1024 == 0 && wend % 1024 == 0 && beta % 1024 == 0 && pa % 1024 == 0 && gh % 1024 == 0 &&
                      pf % 16 == 0,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(total <= 227 * 1024, "shared memory of one CTA");
};

struct DbArgs {
    int L, H;
    long long pos0;
    float scale;
    int dmax;
    const float *Dx;            // D_M table: D_j(pos0 + t) = Dx[t + dmax - Delta_j]
    const int *delta;           // [S]
    int hs_dx, hs_delta;        // per-head strides (0: one shared period)
    const float *lse;           // [BH][L], from the forward
    __nv_bfloat16 *states;      // [BH][nch][2][S][D]: the state entering each chunk
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

__device__ __forceinline__ void fence_proxy_async_global() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

template <int D, int S>
__global__ void __launch_bounds__(kBT, 1)
    k_dchunk_bwd(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                 const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
                 const __grid_constant__ CUtensorMap tm_st,
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
    const int bh = blockIdx.x, hd = bh % a.H;
    const float *Dx = a.Dx + (size_t)hd * a.hs_dx;
    const int L = a.L, nch = (L + kBC - 1) / kBC;
    uint8_t *sQ = dsm + Lay::q, *sK = dsm + Lay::k, *sV = dsm + Lay::v, *sDO = dsm + Lay::dout, *sO = dsm + Lay::o;
    uint8_t *sOst = dsm + Lay::ost, *sK0 = dsm + Lay::k0, *sV0 = dsm + Lay::v0;
    uint8_t *sMuK = dsm + Lay::muk, *sMuV = dsm + Lay::muv, *sW = dsm + Lay::wend, *sBeta = dsm + Lay::beta;
    uint8_t *sPA = dsm + Lay::pa, *sGA = dsm + Lay::ga, *sGm = dsm + Lay::gm, *sGh = dsm + Lay::gh;
    float *sP = reinterpret_cast<float *>(dsm + Lay::pf), *sPV = reinterpret_cast<float *>(dsm + Lay::pvf);
    float *sS = reinterpret_cast<float *>(dsm + Lay::sf), *sDP = reinterpret_cast<float *>(dsm + Lay::dpf);
    float *sD = reinterpret_cast<float *>(dsm + Lay::df), *sAl = reinterpret_cast<float *>(dsm + Lay::af);
    float *sG4 = reinterpret_cast<float *>(dsm + Lay::g4), *sGpre = reinterpret_cast<float *>(dsm + Lay::gpre);
    float *sAend = reinterpret_cast<float *>(dsm + Lay::aend), *sTot = reinterpret_cast<float *>(dsm + Lay::tot);
    int *sdelta = reinterpret_cast<int *>(dsm + Lay::delta);
    float *sLse = reinterpret_cast<float *>(dsm + Lay::lse);
    uint64_t *bar = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    const uint32_t uQ = tc::smem_u32(sQ), uK = tc::smem_u32(sK), uV = tc::smem_u32(sV), uDO = tc::smem_u32(sDO);
    const uint32_t uK0 = tc::smem_u32(sK0), uV0 = tc::smem_u32(sV0), uMuK = tc::smem_u32(sMuK);
    const uint32_t uMuV = tc::smem_u32(sMuV), uW = tc::smem_u32(sW), uBeta = tc::smem_u32(sBeta);
    const uint32_t uPA = tc::smem_u32(sPA), uGA = tc::smem_u32(sGA), uGm = tc::smem_u32(sGm), uGh = tc::smem_u32(sGh);

    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[0], 1);
        tc::mbar_init(&bar[1], 1);
        tc::mbar_init(&bar[2], 1);
        tc::fence_barrier_init();
    }
    for (int j = threadIdx.x; j < S; j += kBT) sdelta[j] = a.delta[(size_t)hd * a.hs_delta + j];
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
    auto load_d = [&](int c) {
        const int t0 = c * kBC, n = min(kBC, L - t0);
        const float *src = Dx + t0 + tu0 + a.dmax - sdelta[tj];
#pragma unroll
        for (int i = 0; i < UPS; ++i) dl[i] = (tu0 + i < n) ? src[i] : 0.f;
    };
    // D_j(u), alpha_j(tau), the sub-block products g and their prefixes Gpre, A_end, Wend and beta
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
        for (int i = 0; i < UPS; ++i) sAl[(tu0 + i) * kBSS + tj] = pre_b * pf[i];
        if (trun == rb0) {
            float gb = tot;
            for (int r2 = trun + 1; r2 < rb0 + RPB; ++r2) gb *= sTot[r2 * S + tj];
            sG4[(trun / RPB) * S + tj] = gb;
            sGpre[(trun / RPB) * S + tj] = pre;
        }
        if (trun == NRUN - 1) sAend[tj] = pre * tot;
        float r = 1.f;
#pragma unroll
        for (int i = UPS - 1; i >= 1; i -= 2) {
            const float w1 = dl[i] * r;
            r -= r * dl[i];
            const float w0 = dl[i - 1] * r;
            r -= r * dl[i - 1];
            st_bf16x2(sW, S, tj, tu0 + i - 1, w0 * suf, w1 * suf);
            st_bf16x2(sBeta, S, tj, tu0 + i - 1, w0 * suf_b, w1 * suf_b);
        }
    };

    // ---- the state (forward sweep) and later its adjoint (reverse sweep), in the accumulator layout
    // of the MMAs that update them: warp w holds NB2 blocks of half kv, row block rb, column blocks cb0..
    const int skv = SMap::kv(warp), sj0 = SMap::rb(warp) * 16, se0 = SMap::cb0(warp) * 16;
    float st[NB2][2][4];
#pragma unroll
    for (int i = 0; i < NB2; ++i)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) st[i][h][q] = 0.f;
    // X <- A_end o X + Wend^T' X_c: A = Wend (rows S), B = the chunk's k or v (kn)
    auto state_update = [&](uint32_t ux, uint32_t uw, bool transposed_a) {
        const float f0 = sAend[sj0 + g8], f1 = sAend[sj0 + g8 + 8];
#pragma unroll
        for (int i = 0; i < NB2; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                st[i][h][0] *= f0; st[i][h][1] *= f0;
                st[i][h][2] *= f1; st[i][h][3] *= f1;
            }
        for (int k0 = 0; k0 < kBC; k0 += 16) {
            uint32_t af[4], b[4];
            if (transposed_a) load_a_t(uw, kBC, sj0, k0, af);
            else load_a(uw, S, sj0, k0, af);
#pragma unroll
            for (int i = 0; i < NB2; ++i) {
                load_b_kn(ux, kBC, se0 + i * 16, k0, b);
                mma16816(st[i][0], af, b[0], b[1]);
                mma16816(st[i][1], af, b[2], b[3]);
            }
        }
    };

    // ================= forward sweep: the state entering every chunk, to the workspace (bf16).  k and
    // v arrive in two stages: (k, v tiles) and (q, dO tiles), which the reverse sweep uses later.
    uint32_t ph0 = 0, ph1 = 0, phs[2] = {0, 0};
    bool ok = true;
    auto issue_kv = [&](int c) {
        const int st2 = c & 1, t0 = c * kBC;
        uint8_t *kb = st2 ? sQ : sK, *vb = st2 ? sDO : sV;
        uint64_t *b = &bar[st2 ? 2 : 0];
        tc::mbar_arrive_expect_tx(b, (uint32_t)(2 * Lay::kTile));
        for (int db = 0; db < D / 64; ++db) {
            tc::tma_load_3d(kb + db * kBC * 128, &tm_k, b, db * 64, t0, bh);
            tc::tma_load_3d(vb + db * kBC * 128, &tm_v, b, db * 64, t0, bh);
        }
    };
    if (nch > 0) {
        load_d(0);
        if (threadIdx.x == 0) issue_kv(0);
    }
    for (int c = 0; c < nch && ok; ++c) {
        const int st2 = c & 1;
        // the other stage was last read by the previous chunk (before the barrier that ended it)
        if (threadIdx.x == 0 && c + 1 < nch) issue_kv(c + 1);
        build_tables();
        if (c + 1 < nch) load_d(c + 1);
        {
            __nv_bfloat16 *dst = a.states + (((size_t)bh * nch + c) * 2 + skv) * S * D;
#pragma unroll
            for (int i = 0; i < NB2; ++i)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int e = se0 + i * 16 + h * 8 + 2 * t4;
                    *reinterpret_cast<uint32_t *>(dst + (size_t)(sj0 + g8) * D + e) = tc::pack_bf16x2(st[i][h][0], st[i][h][1]);
                    *reinterpret_cast<uint32_t *>(dst + (size_t)(sj0 + g8 + 8) * D + e) =
                        tc::pack_bf16x2(st[i][h][2], st[i][h][3]);
                }
        }
        if (!tc::mbar_wait(&bar[st2 ? 2 : 0], phs[st2])) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (17 << 4));
            ok = false;
            break;
        }
        phs[st2] ^= 1;
        state_update(skv ? (st2 ? uDO : uV) : (st2 ? uQ : uK), uW, false);
        __syncthreads();   // the chunk's tiles and tables are read before the next chunk's arrive
    }
    (void)ph0;
    if (!ok) return;
    // the states were written through the generic proxy; the reverse sweep reads them by TMA
    fence_proxy_async_global();
    __syncthreads();

    // ================= reverse sweep
#pragma unroll
    for (int i = 0; i < NB2; ++i)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) st[i][h][q] = 0.f;
    // bf16 copy of the adjoint for the next (earlier) chunk's Wend^T mu
    auto store_mu_copy = [&]() {
        uint8_t *tile = skv ? sMuV : sMuK;
#pragma unroll
        for (int i = 0; i < NB2; ++i)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int e = se0 + i * 16 + h * 8 + 2 * t4;
                st_bf16x2(tile, S, sj0 + g8, e, st[i][h][0], st[i][h][1]);
                st_bf16x2(tile, S, sj0 + g8 + 8, e, st[i][h][2], st[i][h][3]);
            }
    };
    store_mu_copy();
    if (nch > 0) load_d(nch - 1);
    const int sg = threadIdx.x & 15, rp = threadIdx.x >> 4, sb = rp >> 3, ip = rp & 7;
    const unsigned hmask = 0xffffu << (lane & 16);
    for (int c = nch - 1; c >= 0 && ok; --c) {
        const int t0 = c * kBC, n = min(kBC, L - t0);
        if (threadIdx.x == 0) {
            tc::bulk_wait_read0();   // the later chunk's dQ, dK, dV stores have read their staging tiles
            tc::mbar_arrive_expect_tx(&bar[1], (uint32_t)(4 * Lay::kTile + 2 * S * D * 2));
            for (int db = 0; db < D / 64; ++db) {
                const int x = db * 64;
                tc::tma_load_3d(sQ + db * kBC * 128, &tm_q, &bar[1], x, t0, bh);
                tc::tma_load_3d(sK + db * kBC * 128, &tm_k, &bar[1], x, t0, bh);
                tc::tma_load_3d(sV + db * kBC * 128, &tm_v, &bar[1], x, t0, bh);
                tc::tma_load_3d(sDO + db * kBC * 128, &tm_do, &bar[1], x, t0, bh);
                const int srow = (int)((((size_t)bh * nch + c) * 2) * S);
                tc::tma_load_2d(sK0 + db * S * 128, &tm_st, &bar[1], x, srow);
                tc::tma_load_2d(sV0 + db * S * 128, &tm_st, &bar[1], x, srow + S);
            }
        }
        // the chunk before this one (processed next) into L2 meanwhile
        if (threadIdx.x == 0 && c > 0) {
            for (int db = 0; db < D / 64; ++db) {
                const int x = db * 64, tp = t0 - kBC;
                tc::tma_prefetch_3d(&tm_q, x, tp, bh);
                tc::tma_prefetch_3d(&tm_k, x, tp, bh);
                tc::tma_prefetch_3d(&tm_v, x, tp, bh);
                tc::tma_prefetch_3d(&tm_do, x, tp, bh);
            }
            tc::bulk_prefetch_l2(a.states + (((size_t)bh * nch + c - 1) * 2) * S * D, (uint32_t)(2 * S * D * 2));
        }
        if (threadIdx.x < kBC) sLse[threadIdx.x] = threadIdx.x < n ? a.lse[(size_t)bh * L + t0 + threadIdx.x] : 0.f;
        build_tables();
        if (c > 0) load_d(c - 1);
        if (!tc::mbar_wait(&bar[1], ph1)) {
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
                    const uint32_t umu = which == 1 ? uMuK : uMuV;
                    for (int k0 = 0; k0 < kBC; k0 += 16) {
                        load_a_t(ug, kBC, om0, k0, af);
#pragma unroll
                        for (int cb = 0; cb < OCB; ++cb) {
                            load_b_kn(ux, kBC, on0 + cb * 16, k0, b);
                            mma16816(acc[cb][0], af, b[0], b[1]);
                            mma16816(acc[cb][1], af, b[2], b[3]);
                        }
                    }
                    for (int k0 = 0; k0 < S; k0 += 16) {
                        load_a_t(uW, S, om0, k0, af);
#pragma unroll
                        for (int cb = 0; cb < OCB; ++cb) {
                            load_b_kn(umu, S, on0 + cb * 16, k0, b);
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
            // dQ reads K0 and K, dK reads Q and mu_K, dV reads dO and mu_V: none of them reads the v or o
            // tile, which the stores overwrite (V was read by PV, o by delta, before the barriers above)
            out3(0);
            out3(1);
            out3(2);
        }
        // ---- the adjoints of the previous chunk: mu_K <- (g o A)^T Q + A_end o mu_K,
        // mu_V <- (p o A)^T dO + A_end o mu_V (registers; read after dK and dV used the old copies)
        state_update(skv ? uDO : uQ, skv ? uPA : uGA, true);
        tc::fence_proxy_async_smem();
        __syncthreads();
        if (threadIdx.x == 0) {
            for (int db = 0; db < D / 64; ++db) {
                tc::tma_store_3d(&tm_dq, sV + db * kBC * 128, db * 64, t0, bh);
                tc::tma_store_3d(&tm_dk, sO + db * kBC * 128, db * 64, t0, bh);
                tc::tma_store_3d(&tm_dv, sOst + db * kBC * 128, db * 64, t0, bh);
            }
            tc::bulk_commit();
        }
        store_mu_copy();
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
}

template <int D, int S>
cudaError_t launch_dbwd_t(const OpDims &d, const DbArgs &a, const void *q, const void *k, const void *v,
                          const void *dout, void *dq, void *dk, void *dv, cudaStream_t st) {
    CUtensorMap tq, tk, tv, tdo, tst, tdq, tdk, tdv;
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d.L, (uint64_t)d.B * d.H};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d.L * D * 2};
    const uint32_t box[3] = {64, (uint32_t)kBC, 1};
    const int nch = (d.L + kBC - 1) / kBC;
    const uint64_t sdims[2] = {(uint64_t)D, (uint64_t)d.B * d.H * nch * 2 * S};
    const uint64_t sstr[1] = {(uint64_t)D * 2};
    const uint32_t sbox[2] = {64, (uint32_t)S};
    if (!make_tmap_bf16(&tq, q, 3, dims, strides, box) || !make_tmap_bf16(&tk, k, 3, dims, strides, box) ||
        !make_tmap_bf16(&tv, v, 3, dims, strides, box) || !make_tmap_bf16(&tdo, dout, 3, dims, strides, box) ||
        !make_tmap_bf16(&tst, a.states, 2, sdims, sstr, sbox) ||
        !make_tmap_bf16(&tdq, dq, 3, dims, strides, box) || !make_tmap_bf16(&tdk, dk, 3, dims, strides, box) ||
        !make_tmap_bf16(&tdv, dv, 3, dims, strides, box))
        return cudaErrorInvalidValue;
    const int smem = BwLayout<D, S>::total;
    cudaError_t e = cudaFuncSetAttribute(k_dchunk_bwd<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_DECAY, st);
    k_dchunk_bwd<D, S><<<(unsigned)((long long)d.B * d.H), kBT, smem, st>>>(tq, tk, tv, tdo, tst, tdq, tdk, tdv, a);
    return cudaGetLastError();
}

}  // namespace

size_t decay_chunk_bwd_state_bytes(const OpDims &d) {
    const size_t nch = (size_t)(d.L + kBC - 1) / kBC;
    return (size_t)d.B * d.H * nch * 2 * d.S * d.dk * sizeof(__nv_bfloat16);
}

cudaError_t launch_decay_chunk_bwd(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                                   int hs_dx, int hs_delta, const void *q, const void *k, const void *v, const void *o,
                                   const void *dout, const float *lse, void *dq, void *dk, void *dv, void *states,
                                   cudaStream_t st) {
    DbArgs a;
    a.L = d.L; a.H = d.H; a.pos0 = pos0; a.scale = d.scale; a.dmax = dmax;
    a.Dx = Dx; a.delta = delta; a.hs_dx = hs_dx; a.hs_delta = hs_delta;
    a.lse = lse;
    a.states = static_cast<__nv_bfloat16 *>(states);
    a.err = device_error_word();
    if (d.dk == 64) return d.S == 32 ? launch_dbwd_t<64, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                                     : launch_dbwd_t<64, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
    return d.S == 32 ? launch_dbwd_t<128, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                     : launch_dbwd_t<128, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
}

}  // namespace bla
