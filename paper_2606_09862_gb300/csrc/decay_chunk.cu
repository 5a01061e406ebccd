// decay_chunk.cu -- the state-decayed form (Sec. 3.3) in chunks of 32 tokens: forward and
// vector-Jacobian product, bf16 operands, fp32 accumulation.
//
// Per slot j the decayed state is a first-order linear recurrence,
//     X_j(t) = a_j(t) X_j(t-1) + D_j(t) x_t,     a_j(t) = 1 - D_j(t),  D_j(t) = D_M(t - Delta_j),
// for X = K~ (x = k) and X = V~ (x = v).  Over a chunk starting at t0 (tau, u the in-chunk positions),
// with K0, V0 the state entering the chunk,
//     A_j(tau) = prod_{x <= tau} a_j(t0 + x),   W_j(tau, u) = D_j(t0 + u) prod_{u < x <= tau} a_j(t0 + x),
//     s = scale (A o Y + sum_u P o W)  (P = Q K^T, Y = Q K0^T),   p = softmax over the visible slots,
//     o = (p o A) V0 + G V,   G = sum_j p W,
//     K~end = A_end o K0 + Wend K,  V~end = A_end o V0 + Wend V   (Wend[j][u] = W_j(last, u)).
// Every factor is a product of a's: nothing is divided, so the exact zeros of a need no care.
// Given dO and the adjoints mu_K, mu_V of the states at the chunk's end (zero after the last
// chunk: the final state is not differentiated), the chain rule gives, with PV = dO V^T and
// YV = dO V0^T,
//     dp = A o YV + sum_u PV o W,   delta = sum_j p dp,   g = scale p o (dp - delta),
//     G^ = sum_j g W,
//     dQ = (g o A) K0 + G^ K,   dK = G^T Q + Wend^T mu_K,   dV = G^T dO + Wend^T mu_V,
//     mu_K <- (g o A)^T Q + A_end o mu_K,   mu_V <- (p o A)^T dO + A_end o mu_V   (the previous chunk's).
// (A numpy emulation of these lines matched the oracle's decayed VJP to 1e-15.)
//
// Both recurrences are linear with a per-slot diagonal decay, so only thin passes run along the
// sequence; everything else runs one chunk at a time, in parallel over all SMs:
//   1. k_dbtab: per (head, chunk), Wend and A_end for the thin passes and the chains' tables
//      (they depend on the period and the positions only, not on the batch);
//   2. k_dstate: per (head, K~ or V~, 64-column strip), K~_{c+1} = A_end(c) o K~_c + Wend(c) K_c
//      from the entering state: the state entering every chunk, stored in bf16, and the final state;
//   3. forward, k_dfchain: one work item per (head, chunk), each CTA a run of consecutive chunks: s, the
//      softmax and lse, G, then o;
//      backward, k_dbchain: likewise s, p, dp, g, G, G^, then dQ (final), the chunk's own parts G^T Q
//      and G^T dO of dK and dV, and its adjoint contributions Z_K = (g o A)^T Q, Z_V = (p o A)^T dO;
//   4. backward, k_dadj: per (head, strip), from the last chunk back: dK += Wend^T mu_K (dV
//      likewise), then mu <- A_end o mu + Z.
// In the chains the triangle sums (s, dp, G, G^) are split at 16-token sub-blocks: the off-diagonal
// block is a contraction on the tensor cores (W = alpha_j(tau) beta_j(u) across adjacent
// sub-blocks), the diagonal blocks walk u on the CUDA cores.  All contractions are warp-level bf16
// MMAs (m16n8k16).
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

// The chain's tables of one (head, chunk), built by k_dbtab and copied whole into shared memory:
// beta_j(u) (bf16, swizzled [S][64], u < 32 used), D_j(t0 + u) and alpha_j(tau) (fp32 [32][kBSS]),
// and Gpre (fp32 [2][S]: the decay of the sub-blocks before sub-block 0, 1).
template <int S>
struct ChunkTab {
    static constexpr int beta = 0, d = S * 128, alpha = d + kBC * kBSS * 4, gpre = alpha + kBC * kBSS * 4;
    static constexpr int bytes = gpre + 2 * S * 4;
    static_assert(bytes % 16 == 0, "bulk copies move multiples of 16 bytes");
};

// The thin passes' tables of one (head, chunk): Wend (bf16, swizzled [S][64], u < 32 used), then
// A_end (fp32 [S]), one bulk copy.
template <int S>
struct EndTab {
    static constexpr int wend = 0, aend = S * 128, bytes = aend + S * 4;
    static_assert(bytes % 16 == 0, "bulk copies move multiples of 16 bytes");
};

template <int D, int S>
struct BwLayout {
    static constexpr int kTile = kBC * D * 2;          // one [32][D] bf16 tile
    static constexpr int q = 0;                         // bf16 [2][32][D]: q of this item and the next
    static constexpr int dout = q + 2 * kTile;          // bf16 [2][32][D]: dO likewise
    static constexpr int k = dout + 2 * kTile, v = k + kTile;
    static constexpr int o = v + kTile;                 // bf16 [32][D]: dK staging
    static constexpr int ost = o + kTile;               // bf16 [32][D]: dV staging
    static constexpr int k0 = ost + kTile;              // bf16 [S][D]: K~ entering the chunk
    static constexpr int v0 = k0 + S * D * 2;           // bf16 [S][D]: V~ entering the chunk
    static constexpr int zk = v0 + S * D * 2;           // bf16 [S][D]: Z_K staging
    static constexpr int zv = zk + S * D * 2;           // bf16 [S][D]: Z_V staging
    static constexpr int tab = zv + S * D * 2;          // the chunk's tables (ChunkTab)
    static constexpr int pa = tab + ((ChunkTab<S>::bytes + 1023) / 1024) * 1024;   // bf16 [32][64]: p o A
    static constexpr int ga = pa + kBC * 128;           // bf16 [32][64]: g o A
    static constexpr int gm = ga + kBC * 128;           // bf16 [32][64] (u < 32): G
    static constexpr int gh = gm + kBC * 128;           // bf16 [32][64]: G^
    static constexpr int sf = gh + kBC * 128;           // fp32 [32][kBSS]: s, then p, then dQ staging (bf16)
    static constexpr int pf = sf + kBC * kBSS * 4;      // fp32 [32][kBFS]: P
    static constexpr int pvf = pf + kBC * kBFS * 4;     // fp32 [32][kBFS]: PV
    static constexpr int dpf = pvf + kBC * kBFS * 4;    // fp32 [32][kBSS]: dp, then g
    static constexpr int delta = dpf + kBC * kBSS * 4;  // int [S]
    static constexpr int lse = delta + S * 4;           // fp32 [32]
    static constexpr int bars = lse + kBC * 4;          // mbarrier: the item's tiles
    static constexpr int total = bars + 64;
    static_assert(k0 % 1024 == 0 && tab % 1024 == 0 && pa % 1024 == 0 && gh % 1024 == 0 && sf % 1024 == 0 &&
                      kBC * kBSS * 4 >= kTile && pf % 16 == 0,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(total <= 227 * 1024, "shared memory of one CTA");
};

struct DbArgs {
    int L, H, BH;
    int ipc;                    // chain items (chunks) per CTA: CTA b takes items [b ipc, (b + 1) ipc), chunk fastest
    long long pos0;
    float scale;
    int dmax;
    const float *Dx;            // D_M table: D_j(pos0 + t) = Dx[t + dmax - Delta_j]
    const int *delta;           // [S]
    int hs_dx, hs_delta;        // per-head strides (0: one shared period)
    const float *lse;           // [BH][L], from the forward (backward)
    float *lse_out;             // [BH][L] (forward)
    const float *state_in;      // [BH][2][S][D] fp32 or null: the state before the first token (forward)
    float *state_out;           // [BH][2][S][D] fp32 or null: the state after the last token (forward)
    int ntab;                   // heads with their own tables (1 when the heads share one period)
    uint8_t *ctab;              // [ntab][nch] ChunkTab records of the chain
    uint8_t *etab;              // [ntab][nch] EndTab records of the thin passes
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

// N (2 or 4) consecutive 32-bit words of shared memory in one access (16- or 8-byte aligned)
template <typename T, int N>
__device__ __forceinline__ void lds_vec(const T *p, T (&v)[N]) {
    static_assert(N == 2 || N == 4, "vector width");
    if constexpr (N == 4) {
        const uint4 x = *reinterpret_cast<const uint4 *>(p);
        v[0] = __builtin_bit_cast(T, x.x); v[1] = __builtin_bit_cast(T, x.y);
        v[2] = __builtin_bit_cast(T, x.z); v[3] = __builtin_bit_cast(T, x.w);
    } else {
        const uint2 x = *reinterpret_cast<const uint2 *>(p);
        v[0] = __builtin_bit_cast(T, x.x); v[1] = __builtin_bit_cast(T, x.y);
    }
}
template <int N>
__device__ __forceinline__ void sts_vec(float *p, const float (&v)[N]) {
    if constexpr (N == 4) *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    else *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
}
// N bf16 (rounded from fp32) to consecutive columns of a swizzled tile row (within one 16-byte chunk)
template <int N>
__device__ __forceinline__ void st_bf16_vec(uint8_t *p, const float (&v)[N]) {
    if constexpr (N == 4)
        *reinterpret_cast<uint2 *>(p) = make_uint2(tc::pack_bf16x2(v[0], v[1]), tc::pack_bf16x2(v[2], v[3]));
    else *reinterpret_cast<uint32_t *>(p) = tc::pack_bf16x2(v[0], v[1]);
}

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
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (17 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int L = a.L, nch = (L + kBC - 1) / kBC;
    const long long nitems = (long long)a.BH * nch;
    uint8_t *sK = dsm + Lay::k, *sV = dsm + Lay::v, *sO = dsm + Lay::o;
    using Tab = ChunkTab<S>;
    uint8_t *sOst = dsm + Lay::ost, *sK0 = dsm + Lay::k0, *sV0 = dsm + Lay::v0, *sTab = dsm + Lay::tab;
    uint8_t *sZK = dsm + Lay::zk, *sZV = dsm + Lay::zv, *sBeta = sTab + Tab::beta;
    uint8_t *sPA = dsm + Lay::pa, *sGA = dsm + Lay::ga, *sGm = dsm + Lay::gm, *sGh = dsm + Lay::gh;
    float *sP = reinterpret_cast<float *>(dsm + Lay::pf), *sPV = reinterpret_cast<float *>(dsm + Lay::pvf);
    float *sS = reinterpret_cast<float *>(dsm + Lay::sf), *sDP = reinterpret_cast<float *>(dsm + Lay::dpf);
    float *sD = reinterpret_cast<float *>(sTab + Tab::d), *sAl = reinterpret_cast<float *>(sTab + Tab::alpha);
    float *sGpre = reinterpret_cast<float *>(sTab + Tab::gpre);
    int *sdelta = reinterpret_cast<int *>(dsm + Lay::delta);
    float *sLse = reinterpret_cast<float *>(dsm + Lay::lse);
    uint64_t *bar = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    const uint32_t uK = tc::smem_u32(sK), uV = tc::smem_u32(sV);
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
    const int i0 = (int)blockIdx.x * a.ipc, i1 = (int)min(nitems, (long long)i0 + a.ipc);
    // the next item's lse (threads < 32) travels in a register
    float lse_nx = 0.f;
    auto load_lse = [&](int it) {
        const int c = (int)(it % nch), bh = (int)(it / nch), t = c * kBC + (int)threadIdx.x;
        if (threadIdx.x < kBC) lse_nx = t < L ? a.lse[(size_t)bh * L + t] : 0.f;
    };
    auto tab_of = [&](int it) {
        const int tb = a.ntab > 1 ? (int)(it / nch) % a.H : 0;
        return a.ctab + ((size_t)tb * nch + (size_t)(it % nch)) * Tab::bytes;
    };
    // Item it + 1's loads are issued while item it runs, each once its place is free: v, q and dO
    // (the other of the two q / dO buffers) after (a), the tables after (d), k, K0 and V0 after dQ.
    auto issue_vqo = [&](int it, int buf) {
        const int c = (int)(it % nch), bh = (int)(it / nch), t0 = c * kBC;
        tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)(4 * Lay::kTile + 2 * S * D * 2 + Tab::bytes));
        tc::tma_load_4d(sV, &tm_v, &bar[0], 0, t0, 0, bh);
        tc::tma_load_4d(dsm + Lay::q + buf * Lay::kTile, &tm_q, &bar[0], 0, t0, 0, bh);
        tc::tma_load_4d(dsm + Lay::dout + buf * Lay::kTile, &tm_do, &bar[0], 0, t0, 0, bh);
    };
    auto issue_tab = [&](int it) { tc::bulk_load(sTab, tab_of(it), (uint32_t)Tab::bytes, &bar[0]); };
    auto issue_k = [&](int it) {
        const int c = (int)(it % nch), bh = (int)(it / nch);
        const int srow = (int)((((size_t)bh * nch + c) * 2) * S);
        tc::tma_load_4d(sK, &tm_k, &bar[0], 0, c * kBC, 0, bh);
        tc::tma_load_3d(sK0, &tm_st, &bar[0], 0, srow, 0);
        tc::tma_load_3d(sV0, &tm_st, &bar[0], 0, srow + S, 0);
    };
    if (i0 < i1) {
        load_lse(i0);
        if (threadIdx.x == 0) {
            issue_vqo(i0, 0);
            issue_tab(i0);
            issue_k(i0);
        }
    }
    int cur_hd = -1;
    for (int it = i0; it < i1 && ok; ++it) {
        const int c = (int)(it % nch), bh = (int)(it / nch), hd = bh % a.H;
        const int t0 = c * kBC, n = min(kBC, L - t0);
        const int nx = it + 1;
        const int buf = (int)((it - i0) & 1);
        const uint32_t uQ = tc::smem_u32(dsm + Lay::q + buf * Lay::kTile);
        const uint32_t uDO = tc::smem_u32(dsm + Lay::dout + buf * Lay::kTile);
        if (threadIdx.x == kBT - 32 && nx < i1) {
            // the next item's k and states into L2 (their loads follow dQ)
            const int cn = (int)(nx % nch), bn = (int)(nx / nch);
            tc::tma_prefetch_4d(&tm_k, 0, cn * kBC, 0, bn);
            tc::bulk_prefetch_l2(a.states + (((size_t)bn * nch + cn) * 2) * S * D, (uint32_t)(2 * S * D * 2));
        }
        // sdelta and sLse were last read before the previous item's closing barriers
        if (hd != cur_hd) {
            for (int j = threadIdx.x; j < S; j += kBT) sdelta[j] = a.delta[(size_t)hd * a.hs_delta + j];
            cur_hd = hd;
        }
        if (threadIdx.x < kBC) sLse[threadIdx.x] = lse_nx;
        if (nx < i1) load_lse(nx);
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
        // the previous item's stores have read their staging tiles (s, where dQ was staged, is written
        // next; the dK, dV and Z staging tiles later)
        if (threadIdx.x == 0) tc::bulk_wait_read0();
        __syncthreads();
        // v, q and dO are read: the next item's go in (q and dO into the other buffer)
        if (threadIdx.x == 0 && nx < i1) issue_vqo(nx, buf ^ 1);
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
        // Each thread takes rows lo + ip and lo + 15 - ip of its sub-block and walks u down from the
        // sub-block's last token: one load of D_j(u) serves both rows (and both half-warps, which share
        // the sub-block), and P, PV come four tokens at a time.
        {
            const int lo = sb * 16;
            const int rowx[2] = {lo + ip, lo + 15 - ip}, spanx[2] = {ip, 15 - ip};
            float as[2][SPT], ad[2][SPT], r[2][SPT];
#pragma unroll
            for (int x = 0; x < 2; ++x)
#pragma unroll
                for (int k = 0; k < SPT; ++k) { as[x][k] = 0.f; ad[x][k] = 0.f; r[x][k] = 1.f; }
#pragma unroll
            for (int q4 = 3; q4 >= 0; --q4) {
                if (4 * q4 > spanx[1]) continue;
                float pq[2][4], wq[2][4];
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    lds_vec(&sP[rowx[x] * kBFS + lo + 4 * q4], pq[x]);
                    lds_vec(&sPV[rowx[x] * kBFS + lo + 4 * q4], wq[x]);
                }
#pragma unroll
                for (int e = 3; e >= 0; --e) {
                    const int uo = 4 * q4 + e;
                    if (uo > spanx[1]) continue;
                    float dv[SPT];
                    lds_vec(&sD[(lo + uo) * kBSS + sg * SPT], dv);
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        if (uo > spanx[x]) continue;
#pragma unroll
                        for (int k = 0; k < SPT; ++k) {
                            const float w = dv[k] * r[x][k];
                            as[x][k] = fmaf(pq[x][e], w, as[x][k]);
                            ad[x][k] = fmaf(wq[x][e], w, ad[x][k]);
                            r[x][k] = fmaf(-r[x][k], dv[k], r[x][k]);
                        }
                    }
                }
            }
            float pj[2][SPT], dpj[2][SPT], pdp[2] = {0.f, 0.f};
            int dlt[SPT];
            lds_vec(&sdelta[sg * SPT], dlt);
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const int row = rowx[x];
                const long long t = a.pos0 + t0 + row;
                const bool live = row < n;
                const float lr = sLse[row];
                float sv[SPT], dpv[SPT];
                lds_vec(&sS[row * kBSS + sg * SPT], sv);
                lds_vec(&sDP[row * kBSS + sg * SPT], dpv);
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    const float sc = a.scale * (sv[k] + as[x][k]);
                    pj[x][k] = (live && t >= dlt[k]) ? __expf(sc - lr) : 0.f;
                    dpj[x][k] = dpv[k] + ad[x][k];
                    pdp[x] = fmaf(pj[x][k], dpj[x][k], pdp[x]);
                }
            }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                pdp[0] += __shfl_xor_sync(hmask, pdp[0], o);
                pdp[1] += __shfl_xor_sync(hmask, pdp[1], o);
            }
            float gpre[SPT];
            lds_vec(&sGpre[sb * S + sg * SPT], gpre);
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const int row = rowx[x];
                float gj[SPT], al[SPT], pa[SPT], ga[SPT];
                lds_vec(&sAl[row * kBSS + sg * SPT], al);
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    gj[k] = a.scale * pj[x][k] * (dpj[x][k] - pdp[x]);
                    const float A = gpre[k] * al[k];
                    pa[k] = pj[x][k] * A;
                    ga[k] = gj[k] * A;
                }
                sts_vec(&sS[row * kBSS + sg * SPT], pj[x]);
                sts_vec(&sDP[row * kBSS + sg * SPT], gj);
                st_bf16_vec(sPA + sw_off(kBC, row, sg * SPT), pa);
                st_bf16_vec(sGA + sw_off(kBC, row, sg * SPT), ga);
            }
        }
        __syncthreads();
        // ---- (d) G = sum_j p W and G^ = sum_j g W: diagonal sub-blocks by the walk (partials per step in
        // registers, one transposing butterfly over the 16 slot groups each), the block of sub-block 1
        // over sub-block 0 on the tensor cores (warp 0: G, warp 1: G^)
        // (rows lo + ip and lo + 15 - ip walk u down together, as above; the partial sums are kept by u)
        {
            const int lo = sb * 16;
            const int rowx[2] = {lo + ip, lo + 15 - ip}, spanx[2] = {ip, 15 - ip};
            float qv[2][SPT], hv[2][SPT], gp[2][16], hp[2][16];
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                lds_vec(&sS[rowx[x] * kBSS + sg * SPT], qv[x]);
                lds_vec(&sDP[rowx[x] * kBSS + sg * SPT], hv[x]);
            }
#pragma unroll
            for (int uo = 15; uo >= 0; --uo) {
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    gp[x][uo] = 0.f;
                    hp[x][uo] = 0.f;
                }
                if (uo > spanx[1]) continue;
                float dv[SPT];
                lds_vec(&sD[(lo + uo) * kBSS + sg * SPT], dv);
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    if (uo > spanx[x]) continue;
#pragma unroll
                    for (int k = 0; k < SPT; ++k) {
                        gp[x][uo] = fmaf(qv[x][k], dv[k], gp[x][uo]);
                        hp[x][uo] = fmaf(hv[x][k], dv[k], hp[x][uo]);
                        qv[x][k] = fmaf(-qv[x][k], dv[k], qv[x][k]);
                        hv[x][k] = fmaf(-hv[x][k], dv[k], hv[x][k]);
                    }
                }
            }
            // transposing butterfly: slot group sg ends with the row's total at u = lo + sg
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                const bool up = (sg & o) != 0;
#pragma unroll
                for (int i = 0; i < o; ++i)
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        const float s1 = up ? gp[x][i] : gp[x][i + o], m1 = up ? gp[x][i + o] : gp[x][i];
                        const float s2 = up ? hp[x][i] : hp[x][i + o], m2 = up ? hp[x][i + o] : hp[x][i];
                        gp[x][i] = m1 + __shfl_xor_sync(hmask, s1, o);
                        hp[x][i] = m2 + __shfl_xor_sync(hmask, s2, o);
                    }
            }
#pragma unroll
            for (int x = 0; x < 2; ++x)
                if (sg <= spanx[x]) {
                    const uint32_t off = sw_off(kBC, rowx[x], lo + sg);
                    *reinterpret_cast<__nv_bfloat16 *>(sGm + off) = __float2bfloat16_rn(gp[x][0]);
                    *reinterpret_cast<__nv_bfloat16 *>(sGh + off) = __float2bfloat16_rn(hp[x][0]);
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
        // the tables are read: the next item's go in
        if (threadIdx.x == 0 && nx < i1) issue_tab(nx);
        // ---- (e) dQ = (g o A) K0 + G^ K (staged over s), the chunk's parts G^T Q of dK and G^T dO of dV:
        // warp takes row block om0 and OCB column blocks
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
                uint8_t *dst = which == 0 ? reinterpret_cast<uint8_t *>(sS) : which == 1 ? sO : sOst;
#pragma unroll
                for (int cb = 0; cb < OCB; ++cb)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int col = on0 + cb * 16 + h * 8 + 2 * t4;
                        st_bf16x2(dst, kBC, om0 + g8, col, acc[cb][h][0], acc[cb][h][1]);
                        st_bf16x2(dst, kBC, om0 + g8 + 8, col, acc[cb][h][2], acc[cb][h][3]);
                    }
            };
            // dQ first: k, K0 and V0 are then free for the next item
            out3(0);
            tc::fence_proxy_async_smem();
            __syncthreads();
            if (threadIdx.x == 0) {
                tc::tma_store_4d(&tm_dq, sS, 0, t0, 0, bh);
                tc::bulk_commit();
                if (nx < i1) issue_k(nx);
            }
            out3(1);
            out3(2);
        }
        // ---- the chunk's adjoint contributions Z_K = (g o A)^T Q, Z_V = (p o A)^T dO
        z_product(skv ? uDO : uQ, skv ? uPA : uGA);
        {
            uint8_t *tile = skv ? sZV : sZK;
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
            tc::tma_store_4d(&tm_dk, sO, 0, t0, 0, bh);
            tc::tma_store_4d(&tm_dv, sOst, 0, t0, 0, bh);
            tc::tma_store_3d(&tm_z, sZK, 0, srow, 0);
            tc::tma_store_3d(&tm_z, sZV, 0, srow + S, 0);
            tc::bulk_commit();
        }
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
}

// ---- the forward's chunk chains (Sec. 3.3 forward): one work item per (head, 32-token chunk), each CTA
// a run of consecutive chunks, two CTAs per SM.  Per item: P = Q K^T and Y = Q K0^T, the two-level
// triangle sums of s, the softmax over the visible slots (lse written), G = sum_j p W, then
// o = (p o A) V0 + G V, staged over s and stored by TMA.
template <int D, int S>
struct FwLayout {
    static constexpr int kTile = kBC * D * 2;           // one [32][D] bf16 tile
    static constexpr int q = 0, k = q + kTile, v = k + kTile;
    static constexpr int k0 = v + kTile;                // bf16 [S][D]: K~ entering the chunk
    static constexpr int v0 = k0 + S * D * 2;           // bf16 [S][D]: V~ entering the chunk
    static constexpr int tab = v0 + S * D * 2;          // the chunk's tables (ChunkTab)
    static constexpr int pa = tab + ((ChunkTab<S>::bytes + 1023) / 1024) * 1024;   // bf16 [32][64]: p o A
    static constexpr int gm = pa + kBC * 128;           // bf16 [32][64] (u < 32): G
    static constexpr int sf = gm + kBC * 128;           // fp32 [32][kBSS]: s, then p, then o staging (bf16)
    static constexpr int pf = sf + kBC * kBSS * 4;      // fp32 [32][kBFS]: P
    static constexpr int delta = pf + kBC * kBFS * 4;   // int [S]
    static constexpr int bars = delta + S * 4;          // mbarriers: q, k, K0 and tables; v and V0
    static constexpr int total = bars + 64;
    static_assert(k0 % 1024 == 0 && tab % 1024 == 0 && pa % 1024 == 0 && sf % 1024 == 0 && kBC * kBSS * 4 >= kTile,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(2 * (total + 1024) <= 228 * 1024, "two CTAs per SM");
};

template <int D, int S>
__global__ void __launch_bounds__(kBT, 2)
    k_dfchain(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
              const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_st,
              const __grid_constant__ CUtensorMap tm_o, DbArgs a) {
    using Lay = FwLayout<D, S>;
    using Tab = ChunkTab<S>;
    constexpr int SPT = S / 16, SB = S / 16, DB = D / 16, NBLK = 2 + SB;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (19 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int L = a.L, nch = (L + kBC - 1) / kBC;
    const long long nitems = (long long)a.BH * nch;
    uint8_t *sQ = dsm + Lay::q, *sK = dsm + Lay::k, *sV = dsm + Lay::v, *sK0 = dsm + Lay::k0, *sV0 = dsm + Lay::v0;
    uint8_t *sTab = dsm + Lay::tab, *sBeta = sTab + Tab::beta, *sPA = dsm + Lay::pa, *sGm = dsm + Lay::gm;
    float *sS = reinterpret_cast<float *>(dsm + Lay::sf), *sP = reinterpret_cast<float *>(dsm + Lay::pf);
    float *sD = reinterpret_cast<float *>(sTab + Tab::d), *sAl = reinterpret_cast<float *>(sTab + Tab::alpha);
    float *sGpre = reinterpret_cast<float *>(sTab + Tab::gpre);
    int *sdelta = reinterpret_cast<int *>(dsm + Lay::delta);
    uint64_t *bar = reinterpret_cast<uint64_t *>(dsm + Lay::bars);
    const uint32_t uQ = tc::smem_u32(sQ), uK = tc::smem_u32(sK), uV = tc::smem_u32(sV);
    const uint32_t uK0 = tc::smem_u32(sK0), uV0 = tc::smem_u32(sV0), uBeta = tc::smem_u32(sBeta);
    const uint32_t uPA = tc::smem_u32(sPA), uGm = tc::smem_u32(sGm);

    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[0], 1);
        tc::mbar_init(&bar[1], 1);
        tc::fence_barrier_init();
    }
    // the upper triangle of G and the columns past S of p o A stay zero
    for (int i = threadIdx.x; i < kBC * 64 / 2; i += kBT) {
        reinterpret_cast<uint32_t *>(sGm)[i] = 0u;
        reinterpret_cast<uint32_t *>(sPA)[i] = 0u;
    }
    __syncthreads();

    uint32_t ph0 = 0, ph1 = 0;
    bool ok = true;
    const int sg = threadIdx.x & 15, rp = threadIdx.x >> 4, sb = rp >> 3, ip = rp & 7;
    const unsigned hmask = 0xffffu << (lane & 16);
    const int i0 = (int)blockIdx.x * a.ipc, i1 = (int)min(nitems, (long long)i0 + a.ipc);
    auto tab_of = [&](int it) {
        const int tb = a.ntab > 1 ? (it / nch) % a.H : 0;
        return a.ctab + ((size_t)tb * nch + (size_t)(it % nch)) * Tab::bytes;
    };
    // Item it + 1's loads are issued while item it runs, each once its place is free: q, k and K0 after
    // the P/Y products, the tables after G, v and V0 after o.  Barrier 0 covers q, k, K0 and the
    // tables (waited at the item's start), barrier 1 v and V0 (waited before o).
    auto issue_qk = [&](int it) {
        const int c = it % nch, bh = it / nch;
        tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)(2 * Lay::kTile + S * D * 2 + Tab::bytes));
        tc::tma_load_4d(sQ, &tm_q, &bar[0], 0, c * kBC, 0, bh);
        tc::tma_load_4d(sK, &tm_k, &bar[0], 0, c * kBC, 0, bh);
        tc::tma_load_3d(sK0, &tm_st, &bar[0], 0, (int)((((size_t)bh * nch + c) * 2) * S), 0);
    };
    auto issue_tab = [&](int it) { tc::bulk_load(sTab, tab_of(it), (uint32_t)Tab::bytes, &bar[0]); };
    auto issue_v = [&](int it) {
        const int c = it % nch, bh = it / nch;
        tc::mbar_arrive_expect_tx(&bar[1], (uint32_t)(Lay::kTile + S * D * 2));
        tc::tma_load_4d(sV, &tm_v, &bar[1], 0, c * kBC, 0, bh);
        tc::tma_load_3d(sV0, &tm_st, &bar[1], 0, (int)((((size_t)bh * nch + c) * 2 + 1) * S), 0);
    };
    if (i0 < i1 && threadIdx.x == 0) {
        issue_qk(i0);
        issue_tab(i0);
        issue_v(i0);
    }
    int cur_hd = -1;
    for (int it = i0; it < i1 && ok; ++it) {
        const int c = it % nch, bh = it / nch, hd = bh % a.H;
        const int t0 = c * kBC, n = min(kBC, L - t0);
        const int nx = it + 1;
        if (threadIdx.x == kBT - 32 && nx < i1) {
            // the next item's q, k and states into L2 (their loads follow this item's P and Y)
            const int cn = nx % nch, bn = nx / nch;
            tc::tma_prefetch_4d(&tm_q, 0, cn * kBC, 0, bn);
            tc::tma_prefetch_4d(&tm_k, 0, cn * kBC, 0, bn);
            tc::bulk_prefetch_l2(a.states + (((size_t)bn * nch + cn) * 2) * S * D, (uint32_t)(2 * S * D * 2));
        }
        // sdelta was last read before the previous item's closing barriers
        if (hd != cur_hd) {
            for (int j = threadIdx.x; j < S; j += kBT) sdelta[j] = a.delta[(size_t)hd * a.hs_delta + j];
            cur_hd = hd;
        }
        if (!tc::mbar_wait(&bar[0], ph0)) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (19 << 4));
            ok = false;
            break;
        }
        ph0 ^= 1;
        // ---- (a) P = Q K^T and Y = Q K0^T: warp takes row block m0 and column blocks bi and bi + 4 of
        // the row block's 2 + S/16 (blocks 0, 1 are P's, the rest Y's); Y stays in registers
        const int m0 = (warp & 1) * 16, bi = warp >> 1, bt = m0 >> 4;
        const bool has2 = bi + 4 < NBLK;
        float acc0[2][4] = {}, acc1[2][4] = {};
        for (int k0 = 0; k0 < D; k0 += 16) {
            uint32_t af[4], b[4];
            load_a(uQ, kBC, m0, k0, af);
            if (bi < 2) load_b_nk(uK, kBC, bi * 16, k0, b);
            else load_b_nk(uK0, S, (bi - 2) * 16, k0, b);
            mma16816(acc0[0], af, b[0], b[1]);
            mma16816(acc0[1], af, b[2], b[3]);
            if (has2) {
                load_b_nk(uK0, S, (bi + 2) * 16, k0, b);
                mma16816(acc1[0], af, b[0], b[1]);
                mma16816(acc1[1], af, b[2], b[3]);
            }
        }
        if (bi < 2) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int col = bi * 16 + h * 8 + 2 * t4;
                *reinterpret_cast<float2 *>(&sP[(m0 + g8) * kBFS + col]) = make_float2(acc0[h][0], acc0[h][1]);
                *reinterpret_cast<float2 *>(&sP[(m0 + g8 + 8) * kBFS + col]) = make_float2(acc0[h][2], acc0[h][3]);
            }
        }
        // the previous item's o store has read its staging tile (s, written next)
        if (threadIdx.x == 0) tc::bulk_wait_read0();
        __syncthreads();
        // q, k and K0 are read: the next item's go in
        if (threadIdx.x == 0 && nx < i1) issue_qk(nx);
        // ---- (b) the off-diagonal block of sub-block 1 over sub-block 0 (W = alpha beta there), and
        // alpha (Gpre Y + F) into s, for the warp's Y blocks
        auto y_block = [&](int yb, const float (&y)[2][4]) {
            const int n0 = yb * 16;
            float facc[2][4] = {};
            if (bt == 1) {
                const float *p0 = sP + (m0 + g8) * kBFS + 2 * t4, *p1 = p0 + 8 * kBFS;
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
                    sS[row * kBSS + j] = sAl[row * kBSS + j] * fmaf(sGpre[bt * S + j], y[h][q], facc[h][q]);
                }
        };
        if (bi >= 2) y_block(bi - 2, acc0);
        if (has2) y_block(bi + 2, acc1);
        __syncthreads();
        // ---- (c) the diagonal sub-blocks of s on the CUDA cores, then the softmax over the visible
        // slots (the 16 slot groups of a row meet by shuffles), lse, p and p o A.  Each thread takes rows
        // lo + ip and lo + 15 - ip of its sub-block and walks u down from the sub-block's last token:
        // one load of D_j(u) serves both rows and both half-warps, P comes four tokens at a time.
        {
            const int lo = sb * 16;
            const int rowx[2] = {lo + ip, lo + 15 - ip}, spanx[2] = {ip, 15 - ip};
            float as[2][SPT], r[2][SPT];
#pragma unroll
            for (int x = 0; x < 2; ++x)
#pragma unroll
                for (int k = 0; k < SPT; ++k) { as[x][k] = 0.f; r[x][k] = 1.f; }
#pragma unroll
            for (int q4 = 3; q4 >= 0; --q4) {
                if (4 * q4 > spanx[1]) continue;
                float pq[2][4];
#pragma unroll
                for (int x = 0; x < 2; ++x) lds_vec(&sP[rowx[x] * kBFS + lo + 4 * q4], pq[x]);
#pragma unroll
                for (int e = 3; e >= 0; --e) {
                    const int uo = 4 * q4 + e;
                    if (uo > spanx[1]) continue;
                    float dv[SPT];
                    lds_vec(&sD[(lo + uo) * kBSS + sg * SPT], dv);
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        if (uo > spanx[x]) continue;
#pragma unroll
                        for (int k = 0; k < SPT; ++k) {
                            as[x][k] = fmaf(pq[x][e], dv[k] * r[x][k], as[x][k]);
                            r[x][k] = fmaf(-r[x][k], dv[k], r[x][k]);
                        }
                    }
                }
            }
            int dlt[SPT];
            lds_vec(&sdelta[sg * SPT], dlt);
            float sc[2][SPT], mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const long long t = a.pos0 + t0 + rowx[x];
                float sv[SPT];
                lds_vec(&sS[rowx[x] * kBSS + sg * SPT], sv);
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    sc[x][k] = t >= dlt[k] ? a.scale * (sv[k] + as[x][k]) : -INFINITY;
                    mx[x] = fmaxf(mx[x], sc[x][k]);
                }
            }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                mx[0] = fmaxf(mx[0], __shfl_xor_sync(hmask, mx[0], o));
                mx[1] = fmaxf(mx[1], __shfl_xor_sync(hmask, mx[1], o));
            }
            float sum[2] = {0.f, 0.f};
#pragma unroll
            for (int x = 0; x < 2; ++x)
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    sc[x][k] = __expf(sc[x][k] - mx[x]);
                    sum[x] += sc[x][k];
                }
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                sum[0] += __shfl_xor_sync(hmask, sum[0], o);
                sum[1] += __shfl_xor_sync(hmask, sum[1], o);
            }
            float gpre[SPT];
            lds_vec(&sGpre[sb * S + sg * SPT], gpre);
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const int row = rowx[x];
                const float inv = 1.f / sum[x];
                float pj[SPT], al[SPT], pa[SPT];
                lds_vec(&sAl[row * kBSS + sg * SPT], al);
#pragma unroll
                for (int k = 0; k < SPT; ++k) {
                    pj[k] = sc[x][k] * inv;
                    pa[k] = pj[k] * gpre[k] * al[k];
                }
                sts_vec(&sS[row * kBSS + sg * SPT], pj);
                st_bf16_vec(sPA + sw_off(kBC, row, sg * SPT), pa);
                if (sg == 0 && row < n) a.lse_out[(size_t)bh * L + t0 + row] = mx[x] + __logf(sum[x]);
            }
        }
        __syncthreads();
        // ---- (d) G = sum_j p W: the diagonal sub-blocks by the walk (partial sums kept by u, one
        // transposing butterfly over the 16 slot groups), the block of sub-block 1 over sub-block 0 on
        // the tensor cores (warp 0)
        {
            const int lo = sb * 16;
            const int rowx[2] = {lo + ip, lo + 15 - ip}, spanx[2] = {ip, 15 - ip};
            float qv[2][SPT], gp[2][16];
#pragma unroll
            for (int x = 0; x < 2; ++x) lds_vec(&sS[rowx[x] * kBSS + sg * SPT], qv[x]);
#pragma unroll
            for (int uo = 15; uo >= 0; --uo) {
                gp[0][uo] = 0.f;
                gp[1][uo] = 0.f;
                if (uo > spanx[1]) continue;
                float dv[SPT];
                lds_vec(&sD[(lo + uo) * kBSS + sg * SPT], dv);
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    if (uo > spanx[x]) continue;
#pragma unroll
                    for (int k = 0; k < SPT; ++k) {
                        gp[x][uo] = fmaf(qv[x][k], dv[k], gp[x][uo]);
                        qv[x][k] = fmaf(-qv[x][k], dv[k], qv[x][k]);
                    }
                }
            }
            // slot group sg ends with the row's total at u = lo + sg
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1) {
                const bool up = (sg & o) != 0;
#pragma unroll
                for (int i = 0; i < o; ++i)
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        const float s1 = up ? gp[x][i] : gp[x][i + o], m1 = up ? gp[x][i + o] : gp[x][i];
                        gp[x][i] = m1 + __shfl_xor_sync(hmask, s1, o);
                    }
            }
#pragma unroll
            for (int x = 0; x < 2; ++x)
                if (sg <= spanx[x])
                    *reinterpret_cast<__nv_bfloat16 *>(sGm + sw_off(kBC, rowx[x], lo + sg)) =
                        __float2bfloat16_rn(gp[x][0]);
        }
        if (warp == 0) {
            float acc[2][4] = {};
#pragma unroll
            for (int kk = 0; kk < SB; ++kk) {
                float xv[2][2][2];
#pragma unroll
                for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                    for (int e = 0; e < 2; ++e)
#pragma unroll
                        for (int rh = 0; rh < 2; ++rh) {
                            const int row = 16 + g8 + rh * 8, j = kk * 16 + ch * 8 + 2 * t4 + e;
                            xv[rh][ch][e] = sS[row * kBSS + j] * sAl[row * kBSS + j];
                        }
                const uint32_t af[4] = {tc::pack_bf16x2(xv[0][0][0], xv[0][0][1]),
                                        tc::pack_bf16x2(xv[1][0][0], xv[1][0][1]),
                                        tc::pack_bf16x2(xv[0][1][0], xv[0][1][1]),
                                        tc::pack_bf16x2(xv[1][1][0], xv[1][1][1])};
                uint32_t b[4];
                load_b_kn(uBeta, S, 0, kk * 16, b);
                mma16816(acc[0], af, b[0], b[1]);
                mma16816(acc[1], af, b[2], b[3]);
            }
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int col = h * 8 + 2 * t4;
                st_bf16x2(sGm, kBC, 16 + g8, col, acc[h][0], acc[h][1]);
                st_bf16x2(sGm, kBC, 24 + g8, col, acc[h][2], acc[h][3]);
            }
        }
        __syncthreads();
        // the tables are read: the next item's go in
        if (threadIdx.x == 0 && nx < i1) issue_tab(nx);
        // ---- (e) o = (p o A) V0 + G V, staged over s: warp takes row block om0 and OCB column blocks
        if (!tc::mbar_wait(&bar[1], ph1)) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (19 << 4));
            ok = false;
            break;
        }
        ph1 ^= 1;
        {
            constexpr int OCB = DB / 4;
            const int om0 = (warp & 1) * 16, on0 = (warp >> 1) * OCB * 16;
            float acc[OCB][2][4] = {};
            uint32_t af[4], b[4];
            for (int k0 = 0; k0 < S; k0 += 16) {
                load_a(uPA, kBC, om0, k0, af);
#pragma unroll
                for (int cb = 0; cb < OCB; ++cb) {
                    load_b_kn(uV0, S, on0 + cb * 16, k0, b);
                    mma16816(acc[cb][0], af, b[0], b[1]);
                    mma16816(acc[cb][1], af, b[2], b[3]);
                }
            }
            for (int k0 = 0; k0 < kBC; k0 += 16) {
                load_a(uGm, kBC, om0, k0, af);
#pragma unroll
                for (int cb = 0; cb < OCB; ++cb) {
                    load_b_kn(uV, kBC, on0 + cb * 16, k0, b);
                    mma16816(acc[cb][0], af, b[0], b[1]);
                    mma16816(acc[cb][1], af, b[2], b[3]);
                }
            }
            uint8_t *dst = reinterpret_cast<uint8_t *>(sS);
#pragma unroll
            for (int cb = 0; cb < OCB; ++cb)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int col = on0 + cb * 16 + h * 8 + 2 * t4;
                    st_bf16x2(dst, kBC, om0 + g8, col, acc[cb][h][0], acc[cb][h][1]);
                    st_bf16x2(dst, kBC, om0 + g8 + 8, col, acc[cb][h][2], acc[cb][h][3]);
                }
        }
        tc::fence_proxy_async_smem();
        __syncthreads();
        if (threadIdx.x == 0) {
            tc::tma_store_4d(&tm_o, sS, 0, t0, 0, bh);
            tc::bulk_commit();
            if (nx < i1) issue_v(nx);   // v and V0 are read
        }
    }
    if (threadIdx.x == 0) tc::bulk_wait0();
}

// ---- the tables of every (head, chunk), one thread per slot j: Wend and A_end for the thin passes,
// and the chain's ChunkTab record (D, alpha, beta, Gpre).  D_j(t0 + u) = Dx[t0 + u + dmax - Delta_j];
// tokens past L contribute nothing (D = 0).
template <int S>
__global__ void __launch_bounds__(S) k_dbtab(DbArgs a) {
    using Tab = ChunkTab<S>;
    const int c = blockIdx.x, h = blockIdx.y, j = threadIdx.x, nch = (a.L + kBC - 1) / kBC;
    const int t0 = c * kBC, n = min(kBC, a.L - t0);
    const float *src = a.Dx + (size_t)h * a.hs_dx + t0 + a.dmax - a.delta[(size_t)h * a.hs_delta + j];
    const size_t ti = (size_t)h * nch + c;
    uint8_t *w = a.etab + ti * EndTab<S>::bytes + EndTab<S>::wend;
    uint8_t *rec = a.ctab + ti * Tab::bytes;
    float *rd = reinterpret_cast<float *>(rec + Tab::d), *ral = reinterpret_cast<float *>(rec + Tab::alpha);
    float *rg = reinterpret_cast<float *>(rec + Tab::gpre);
    float dv[kBC];
#pragma unroll
    for (int u = 0; u < kBC; ++u) {
        dv[u] = u < n ? src[u] : 0.f;
        rd[u * kBSS + j] = dv[u];
        for (int col = S + j; col < kBSS; col += S) rd[u * kBSS + col] = 0.f, ral[u * kBSS + col] = 0.f;
    }
    // alpha_j(tau): the decay from the start of tau's 16-token sub-block through tau; Gpre: before it
    float p = 1.f;
    rg[j] = 1.f;
#pragma unroll
    for (int u = 0; u < kBC; ++u) {
        if (u == 16) {
            rg[S + j] = p;
            p = 1.f;
        }
        p *= 1.f - dv[u];
        ral[u * kBSS + j] = p;
    }
    // Wend_j(u) = D_j(u) x the decay after u to the chunk's end; beta_j(u) the same to the end of u's
    // sub-block
    float r = 1.f, rb = 1.f;
#pragma unroll
    for (int u = kBC - 2; u >= 0; u -= 2) {
        if (u == 14) rb = 1.f;
        const float d1 = dv[u + 1], d0 = dv[u];
        const float w1 = d1 * r;
        r -= r * d1;
        const float w0 = d0 * r;
        r -= r * d0;
        const float b1 = d1 * rb;
        rb -= rb * d1;
        const float b0 = d0 * rb;
        rb -= rb * d0;
        *reinterpret_cast<uint32_t *>(w + wmma16::sw_off(S, j, u)) = tc::pack_bf16x2(w0, w1);
        *reinterpret_cast<uint32_t *>(rec + Tab::beta + wmma16::sw_off(S, j, u)) = tc::pack_bf16x2(b0, b1);
    }
    for (int u = kBC; u < 64; u += 2) {
        *reinterpret_cast<uint32_t *>(w + wmma16::sw_off(S, j, u)) = 0u;
        *reinterpret_cast<uint32_t *>(rec + Tab::beta + wmma16::sw_off(S, j, u)) = 0u;
    }
    reinterpret_cast<float *>(a.etab + ti * EndTab<S>::bytes + EndTab<S>::aend)[j] = r;
}

// ---- the thin passes along the sequence.  One CTA per (64-column strip, K~ or V~, head): compute
// warps that never wait for one another, and a producer warp that keeps kNS stages of loads in
// flight (a stage is released when every compute warp has arrived on its empty barrier).
constexpr int kNS = 4;           // pipeline stages

template <int S>
struct ThinLayout {
    static constexpr int kT = kBC * 128;                    // [32][64] bf16 tile
    static constexpr int kW = S * 128;                      // [S][64] bf16 tile
    // a stage: Z (adjoint pass only) | k, v, dK or dV | the EndTab record, in whole 1024-byte blocks
    static constexpr int stage = ((kW + kT + EndTab<S>::bytes) + 1023) / 1024 * 1024;
    static constexpr int mu = kNS * stage;                  // bf16 [S][64]: mu (adjoint pass)
    static constexpr int out = mu + kW;                     // per compute warp two 2 KB staging tiles
    static constexpr int bars = out + 4 * 2 * 2048;         // full[kNS], empty[kNS]
    static constexpr int total = bars + 16 * kNS;
    static_assert(stage % 1024 == 0 && mu % 1024 == 0 && out % 1024 == 0, "swizzled tiles need 1024-byte alignment");
};

// K~_{c+1} = A_end(c) o K~_c + Wend(c) K_c from the entering state (or zero): the state entering every
// chunk goes to `states` (bf16), the final one to state_out.  Compute warp w owns rows 16 w .. 16 w + 15
// of the strip (S / 16 warps); each stores its rows of every chunk's state by its own TMA store.
template <int D, int S>
__global__ void __launch_bounds__((S / 16 + 1) * 32)
    k_dstate(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
             const __grid_constant__ CUtensorMap tm_st16, DbArgs a) {
    using Lay = ThinLayout<S>;
    constexpr int NW = S / 16;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (18 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int strip = blockIdx.x, kv = blockIdx.y, bh = blockIdx.z;
    const int tab = a.ntab > 1 ? bh % a.H : 0;
    const int nch = (a.L + kBC - 1) / kBC, x = strip * 64;
    uint64_t *full = reinterpret_cast<uint64_t *>(dsm + Lay::bars), *empty = full + kNS;
    auto sx = [&](int s) { return dsm + s * Lay::stage + Lay::kW; };
    auto sw = [&](int s) { return dsm + s * Lay::stage + Lay::kW + Lay::kT + EndTab<S>::wend; };
    auto sa = [&](int s) {
        return reinterpret_cast<const float *>(dsm + s * Lay::stage + Lay::kW + Lay::kT + EndTab<S>::aend);
    };
    if (threadIdx.x == 0) {
        for (int s = 0; s < kNS; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], NW);
        }
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (warp == NW) {
        // producer: chunk i into stage i % kNS once the compute warps have released it
        if (lane == 0) {
            const CUtensorMap *tx = kv ? &tm_v : &tm_k;
            for (int i = 0; i < nch; ++i) {
                const int s = i % kNS;
                if (i >= kNS && !tc::mbar_wait(&empty[s], (uint32_t)((i / kNS - 1) & 1))) {
                    report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (18 << 4));
                    break;
                }
                tc::mbar_arrive_expect_tx(&full[s], (uint32_t)(Lay::kT + EndTab<S>::bytes));
                tc::tma_load_3d(sx(s), tx, &full[s], x, i * kBC, bh);
                tc::bulk_load(sw(s), a.etab + ((size_t)tab * nch + i) * EndTab<S>::bytes, (uint32_t)EndTab<S>::bytes,
                              &full[s]);
            }
        }
        return;
    }
    const int r0 = warp * 16;
    float acc[4][2][4];
    // the warp's rows of an fp32 [BH][2][S][D] state: acc element (b, h, q) is row r0 + g8 + 8 (q >> 1),
    // column x + 16 b + 8 h + 2 t4 + (q & 1)
    auto state_at = [&](int rh) { return ((size_t)(bh * 2 + kv) * S + r0 + g8 + 8 * rh) * D + x + 2 * t4; };
#pragma unroll
    for (int b = 0; b < 4; ++b)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int rh = 0; rh < 2; ++rh) {
                float2 v0 = make_float2(0.f, 0.f);
                if (a.state_in) v0 = *reinterpret_cast<const float2 *>(a.state_in + state_at(rh) + b * 16 + h * 8);
                acc[b][h][2 * rh] = v0.x;
                acc[b][h][2 * rh + 1] = v0.y;
            }
    uint8_t *stg = dsm + Lay::out + warp * 2 * 2048;
    bool ok = true;
    for (int i = 0; i < nch; ++i) {
        const int s = i % kNS, ob = i & 1;
        // the state entering chunk i: the warp's 16 rows, by its own store
        if (lane == 0) tc::bulk_wait_read1();   // the store from staging tile ob two chunks ago has read it
        __syncwarp();
        uint8_t *tile = stg + ob * 2048;
#pragma unroll
        for (int b = 0; b < 4; ++b)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int col = b * 16 + h * 8 + 2 * t4;
                st_bf16x2(tile, 16, g8, col, acc[b][h][0], acc[b][h][1]);
                st_bf16x2(tile, 16, g8 + 8, col, acc[b][h][2], acc[b][h][3]);
            }
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            tc::tma_store_2d(&tm_st16, tile, x, (int)((((size_t)bh * nch + i) * 2 + kv) * S + r0));
            tc::bulk_commit();
        }
        if (!tc::mbar_wait(&full[s], (uint32_t)((i / kNS) & 1))) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (18 << 4));
            ok = false;
            break;
        }
        // acc <- A_end o acc + Wend K_i: A = the Wend rows r0.. (tokens as K), B = the chunk's strip
        const float *ae = sa(s);
        const float f0 = ae[r0 + g8], f1 = ae[r0 + g8 + 8];
#pragma unroll
        for (int b = 0; b < 4; ++b)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                acc[b][h][0] *= f0; acc[b][h][1] *= f0;
                acc[b][h][2] *= f1; acc[b][h][3] *= f1;
            }
        const uint32_t uW = tc::smem_u32(sw(s)), uX = tc::smem_u32(sx(s));
#pragma unroll
        for (int k0 = 0; k0 < kBC; k0 += 16) {
            uint32_t af[4], bf[4];
            load_a(uW, S, r0, k0, af);
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                load_b_kn(uX, kBC, b * 16, k0, bf);
                mma16816(acc[b][0], af, bf[0], bf[1]);
                mma16816(acc[b][1], af, bf[2], bf[3]);
            }
        }
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&empty[s]);
    }
    if (ok && a.state_out) {
#pragma unroll
        for (int b = 0; b < 4; ++b)
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int rh = 0; rh < 2; ++rh)
                    *reinterpret_cast<float2 *>(a.state_out + state_at(rh) + b * 16 + h * 8) =
                        make_float2(acc[b][h][2 * rh], acc[b][h][2 * rh + 1]);
    }
    if (lane == 0) tc::bulk_wait0();
}

// From the last chunk back: dK_c += Wend(c)^T mu_c (a bf16 copy of mu as the MMA operand), then
// mu_{c-1} = A_end(c) o mu_c + Z_c.  Compute warp w (4 of them) owns columns 16 w .. 16 w + 15 of the
// strip for all S rows of mu, so the contraction over the slots needs no other warp's data; each
// stores its [32][16] block of dK by its own TMA store (unswizzled box).
template <int D, int S>
__global__ void __launch_bounds__(5 * 32)
    k_dadj(const __grid_constant__ CUtensorMap tm_dk, const __grid_constant__ CUtensorMap tm_dv,
           const __grid_constant__ CUtensorMap tm_dk16, const __grid_constant__ CUtensorMap tm_dv16,
           const __grid_constant__ CUtensorMap tm_z, DbArgs a) {
    using Lay = ThinLayout<S>;
    constexpr int NW = 4, SB = S / 16;
    extern __shared__ __align__(1024) uint8_t dsm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g8 = lane >> 2, t4 = lane & 3;
    if (tc::smem_u32(dsm) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (18 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    const int strip = blockIdx.x, kv = blockIdx.y, bh = blockIdx.z;
    const int tab = a.ntab > 1 ? bh % a.H : 0;
    const int nch = (a.L + kBC - 1) / kBC, x = strip * 64;
    uint64_t *full = reinterpret_cast<uint64_t *>(dsm + Lay::bars), *empty = full + kNS;
    auto sz = [&](int s) { return dsm + s * Lay::stage; };
    auto sx = [&](int s) { return dsm + s * Lay::stage + Lay::kW; };
    auto sw = [&](int s) { return dsm + s * Lay::stage + Lay::kW + Lay::kT + EndTab<S>::wend; };
    auto sa = [&](int s) {
        return reinterpret_cast<const float *>(dsm + s * Lay::stage + Lay::kW + Lay::kT + EndTab<S>::aend);
    };
    if (threadIdx.x == 0) {
        for (int s = 0; s < kNS; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], NW);
        }
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (warp == NW) {
        // producer: step i (chunk nch - 1 - i) into stage i % kNS: Z, the chain's dK (or dV) part, EndTab
        if (lane == 0) {
            const CUtensorMap *tx = kv ? &tm_dv : &tm_dk;
            for (int i = 0; i < nch; ++i) {
                const int s = i % kNS, c = nch - 1 - i;
                if (i >= kNS && !tc::mbar_wait(&empty[s], (uint32_t)((i / kNS - 1) & 1))) {
                    report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (18 << 4));
                    break;
                }
                tc::mbar_arrive_expect_tx(&full[s], (uint32_t)(Lay::kW + Lay::kT + EndTab<S>::bytes));
                tc::tma_load_2d(sz(s), &tm_z, &full[s], x, (int)((((size_t)bh * nch + c) * 2 + kv) * S));
                tc::tma_load_3d(sx(s), tx, &full[s], x, c * kBC, bh);
                tc::bulk_load(sw(s), a.etab + ((size_t)tab * nch + c) * EndTab<S>::bytes, (uint32_t)EndTab<S>::bytes,
                              &full[s]);
            }
        }
        return;
    }
    const int n0 = warp * 16;
    const CUtensorMap *tout = kv ? &tm_dv16 : &tm_dk16;
    float mu[SB][2][4];
#pragma unroll
    for (int rb = 0; rb < SB; ++rb)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int q = 0; q < 4; ++q) mu[rb][h][q] = 0.f;
    uint8_t *sMu = dsm + Lay::mu;
    const uint32_t uMu = tc::smem_u32(sMu);
    __nv_bfloat16 *stg = reinterpret_cast<__nv_bfloat16 *>(dsm + Lay::out + warp * 2 * 2048);
    for (int i = 0; i < nch; ++i) {
        const int s = i % kNS, c = nch - 1 - i, ob = i & 1;
        if (!tc::mbar_wait(&full[s], (uint32_t)((i / kNS) & 1))) {
            report_device_error(a.err, DEVERR_MBAR_TIMEOUT | (18 << 4));
            break;
        }
        if (i > 0) {   // mu is zero after the last chunk
            // the warp's columns of mu in bf16, as the B operand
#pragma unroll
            for (int rb = 0; rb < SB; ++rb)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int col = n0 + h * 8 + 2 * t4;
                    st_bf16x2(sMu, S, rb * 16 + g8, col, mu[rb][h][0], mu[rb][h][1]);
                    st_bf16x2(sMu, S, rb * 16 + g8 + 8, col, mu[rb][h][2], mu[rb][h][3]);
                }
            __syncwarp();
            float o[2][2][4] = {};
            const uint32_t uW = tc::smem_u32(sw(s));
#pragma unroll
            for (int k0 = 0; k0 < S; k0 += 16) {
                uint32_t bf[4];
                load_b_kn(uMu, S, n0, k0, bf);
#pragma unroll
                for (int tb = 0; tb < 2; ++tb) {
                    uint32_t af[4];
                    load_a_t(uW, S, tb * 16, k0, af);
                    mma16816(o[tb][0], af, bf[0], bf[1]);
                    mma16816(o[tb][1], af, bf[2], bf[3]);
                }
            }
            // + the chain's part, into the warp's dense [32][16] staging tile
            if (lane == 0) tc::bulk_wait_read1();
            __syncwarp();
            __nv_bfloat16 *tile = stg + ob * (kBC * 16);
            const uint8_t *dk = sx(s);
#pragma unroll
            for (int tb = 0; tb < 2; ++tb)
#pragma unroll
                for (int h = 0; h < 2; ++h)
#pragma unroll
                    for (int rh = 0; rh < 2; ++rh) {
                        const int row = tb * 16 + g8 + rh * 8, cl = h * 8 + 2 * t4;
                        const float2 l = __bfloat1622float2(
                            *reinterpret_cast<const __nv_bfloat162 *>(dk + sw_off(kBC, row, n0 + cl)));
                        *reinterpret_cast<uint32_t *>(tile + row * 16 + cl) =
                            tc::pack_bf16x2(o[tb][h][2 * rh] + l.x, o[tb][h][2 * rh + 1] + l.y);
                    }
            tc::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                tc::tma_store_3d(tout, tile, x + n0, c * kBC, bh);
                tc::bulk_commit();
            }
        }
        // mu <- A_end o mu + Z_c
        const float *ae = sa(s);
        const uint8_t *z = sz(s);
#pragma unroll
        for (int rb = 0; rb < SB; ++rb) {
            const float f0 = ae[rb * 16 + g8], f1 = ae[rb * 16 + g8 + 8];
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int rh = 0; rh < 2; ++rh) {
                    const int row = rb * 16 + g8 + rh * 8, col = n0 + h * 8 + 2 * t4;
                    const float2 zz =
                        __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(z + sw_off(S, row, col)));
                    const float f = rh ? f1 : f0;
                    mu[rb][h][2 * rh] = fmaf(f, mu[rb][h][2 * rh], zz.x);
                    mu[rb][h][2 * rh + 1] = fmaf(f, mu[rb][h][2 * rh + 1], zz.y);
                }
        }
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&empty[s]);
    }
    if (lane == 0) tc::bulk_wait0();
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
    // the thin passes: [32][64] strips of k, v and of the chain's dK, dV parts, [16][64] blocks of the
    // states (one per warp), [S][64] strips of Z, and the [32][16] blocks of dK and dV each warp stores
    CUtensorMap tk, tv, tst16, tz, tdk, tdv, tdk16, tdv16;
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d.L, (uint64_t)d.B * d.H};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d.L * D * 2};
    const uint32_t box[3] = {64, (uint32_t)kBC, 1}, box16[3] = {16, (uint32_t)kBC, 1};
    const int nch = (d.L + kBC - 1) / kBC;
    const uint64_t sdims[2] = {(uint64_t)D, (uint64_t)d.B * d.H * nch * 2 * S};
    const uint64_t sstr[1] = {(uint64_t)D * 2};
    const uint32_t sbox[2] = {64, (uint32_t)S}, sbox16[2] = {64, 16};
    if (!make_tmap_bf16(&tk, k, 3, dims, strides, box) || !make_tmap_bf16(&tv, v, 3, dims, strides, box) ||
        !make_tmap_bf16(&tst16, a.states, 2, sdims, sstr, sbox16) ||
        !make_tmap_bf16(&tz, a.zbuf, 2, sdims, sstr, sbox) || !make_tmap_bf16(&tdk, dk, 3, dims, strides, box) ||
        !make_tmap_bf16(&tdv, dv, 3, dims, strides, box) ||
        !make_tmap_bf16(&tdk16, dk, 3, dims, strides, box16, false) ||
        !make_tmap_bf16(&tdv16, dv, 3, dims, strides, box16, false))
        return cudaErrorInvalidValue;
    // the chain moves whole [32][D] and [S][D] tiles in one copy each: the 64-column blocks are a
    // further dimension of the maps (128 bytes apart), so a box lands as [D / 64][rows][64]
    CUtensorMap cq, ck, cv, cdo, cst, cz, cdq, cdk, cdv;
    const uint64_t cdims[4] = {64, (uint64_t)d.L, (uint64_t)(D / 64), (uint64_t)d.B * d.H};
    const uint64_t cstr[3] = {(uint64_t)D * 2, 128, (uint64_t)d.L * D * 2};
    const uint32_t cbox[4] = {64, (uint32_t)kBC, (uint32_t)(D / 64), 1};
    const uint64_t csdims[3] = {64, (uint64_t)d.B * d.H * nch * 2 * S, (uint64_t)(D / 64)};
    const uint64_t csstr[2] = {(uint64_t)D * 2, 128};
    const uint32_t csbox[3] = {64, (uint32_t)S, (uint32_t)(D / 64)};
    if (!make_tmap_bf16(&cq, q, 4, cdims, cstr, cbox) || !make_tmap_bf16(&ck, k, 4, cdims, cstr, cbox) ||
        !make_tmap_bf16(&cv, v, 4, cdims, cstr, cbox) || !make_tmap_bf16(&cdo, dout, 4, cdims, cstr, cbox) ||
        !make_tmap_bf16(&cst, a.states, 3, csdims, csstr, csbox) ||
        !make_tmap_bf16(&cz, a.zbuf, 3, csdims, csstr, csbox) || !make_tmap_bf16(&cdq, dq, 4, cdims, cstr, cbox) ||
        !make_tmap_bf16(&cdk, dk, 4, cdims, cstr, cbox) || !make_tmap_bf16(&cdv, dv, 4, cdims, cstr, cbox))
        return cudaErrorInvalidValue;
    const int smem = BwLayout<D, S>::total, ssm = ThinLayout<S>::total;
    cudaError_t e = cudaFuncSetAttribute(k_dbchain<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_dstate<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, ssm);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_dadj<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, ssm);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_DECAY, st);
    k_dbtab<S><<<dim3((unsigned)nch, (unsigned)a.ntab), S, 0, st>>>(a);
    const dim3 sgrid((unsigned)(D / 64), 2u, (unsigned)a.BH);
    k_dstate<D, S><<<sgrid, (S / 16 + 1) * 32, ssm, st>>>(tk, tv, tst16, a);
    const long long items = (long long)a.BH * nch;
    if (items > 0x7fffffffLL) return cudaErrorInvalidValue;   // the chain indexes its items in 32 bits
    DbArgs ac = a;
    ac.ipc = (int)((items + sm_count_db() - 1) / sm_count_db());
    const int grid = (int)((items + ac.ipc - 1) / ac.ipc);
    k_dbchain<D, S><<<(unsigned)grid, kBT, smem, st>>>(cq, ck, cv, cdo, cst, cz, cdq, cdk, cdv, ac);
    k_dadj<D, S><<<sgrid, 5 * 32, ssm, st>>>(tdk, tdv, tdk16, tdv16, tz, a);
    return cudaGetLastError();
}

// the pieces of the backward's workspace: states, Z, Wend tables, A_end tables
struct DbWs {
    size_t states, z, etab, ctab, total;
};

DbWs db_ws(const OpDims &d, bool with_z) {
    const size_t nch = (size_t)(d.L + kBC - 1) / kBC, ntab = d.periods ? (size_t)d.H : 1;
    const size_t per = align_up((size_t)d.B * d.H * nch * 2 * d.S * d.dk * sizeof(__nv_bfloat16), 256);
    DbWs w;
    w.states = 0;
    w.z = per;
    w.etab = with_z ? 2 * per : per;
    const size_t end_bytes = d.S == 32 ? (size_t)EndTab<32>::bytes : (size_t)EndTab<64>::bytes;
    w.ctab = w.etab + align_up(ntab * nch * end_bytes, 256);
    const size_t tab_bytes = d.S == 32 ? (size_t)ChunkTab<32>::bytes : (size_t)ChunkTab<64>::bytes;
    w.total = w.ctab + align_up(ntab * nch * tab_bytes, 256);
    return w;
}

template <int D, int S>
cudaError_t launch_dfwd_t(const OpDims &d, const DbArgs &a, const void *q, const void *k, const void *v, void *o,
                          cudaStream_t st) {
    CUtensorMap tk, tv, tst16, cq, ck, cv, cst, co;
    const int nch = (d.L + kBC - 1) / kBC;
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d.L, (uint64_t)d.B * d.H};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d.L * D * 2};
    const uint32_t box[3] = {64, (uint32_t)kBC, 1};
    const uint64_t sdims[2] = {(uint64_t)D, (uint64_t)d.B * d.H * nch * 2 * S};
    const uint64_t sstr[1] = {(uint64_t)D * 2};
    const uint32_t sbox16[2] = {64, 16};
    const uint64_t cdims[4] = {64, (uint64_t)d.L, (uint64_t)(D / 64), (uint64_t)d.B * d.H};
    const uint64_t cstr[3] = {(uint64_t)D * 2, 128, (uint64_t)d.L * D * 2};
    const uint32_t cbox[4] = {64, (uint32_t)kBC, (uint32_t)(D / 64), 1};
    const uint64_t csdims[3] = {64, (uint64_t)d.B * d.H * nch * 2 * S, (uint64_t)(D / 64)};
    const uint64_t csstr[2] = {(uint64_t)D * 2, 128};
    const uint32_t csbox[3] = {64, (uint32_t)S, (uint32_t)(D / 64)};
    if (!make_tmap_bf16(&tk, k, 3, dims, strides, box) || !make_tmap_bf16(&tv, v, 3, dims, strides, box) ||
        !make_tmap_bf16(&tst16, a.states, 2, sdims, sstr, sbox16) || !make_tmap_bf16(&cq, q, 4, cdims, cstr, cbox) ||
        !make_tmap_bf16(&ck, k, 4, cdims, cstr, cbox) || !make_tmap_bf16(&cv, v, 4, cdims, cstr, cbox) ||
        !make_tmap_bf16(&cst, a.states, 3, csdims, csstr, csbox) || !make_tmap_bf16(&co, o, 4, cdims, cstr, cbox))
        return cudaErrorInvalidValue;
    const int smem = FwLayout<D, S>::total, ssm = ThinLayout<S>::total;
    cudaError_t e = cudaFuncSetAttribute(k_dfchain<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_dstate<D, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, ssm);
    if (e != cudaSuccess) return e;
    const long long items = (long long)a.BH * nch;
    if (items > 0x7fffffffLL) return cudaErrorInvalidValue;   // the chain indexes its items in 32 bits
    ProfScope ps(BLA_K_DECAY, st);
    k_dbtab<S><<<dim3((unsigned)nch, (unsigned)a.ntab), S, 0, st>>>(a);
    k_dstate<D, S><<<dim3((unsigned)(D / 64), 2u, (unsigned)a.BH), (S / 16 + 1) * 32, ssm, st>>>(tk, tv, tst16, a);
    DbArgs ac = a;
    const long long slots = 2LL * sm_count_db();   // two chain CTAs per SM
    ac.ipc = (int)((items + slots - 1) / slots);
    const int grid = (int)((items + ac.ipc - 1) / ac.ipc);
    k_dfchain<D, S><<<(unsigned)grid, kBT, smem, st>>>(cq, ck, cv, cst, co, ac);
    return cudaGetLastError();
}

}  // namespace

size_t decay_chunk_bwd_ws_bytes(const OpDims &d) { return db_ws(d, true).total; }
size_t decay_chunk_fwd_ws_bytes(const OpDims &d) { return db_ws(d, false).total; }

bool decay_chunk_supported(const OpDims &d) {
    // (the thin passes put the heads on the grid's z dimension: at most 65535 of them)
    return d.dtype == BLA_BF16 && d.dk == d.dv && (d.dk == 64 || d.dk == 128) && (d.S == 32 || d.S == 64) &&
           d.L > 0 && (long long)d.B * d.H <= 65535;
}

cudaError_t launch_decay_chunk_bwd(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                                   int hs_dx, int hs_delta, const void *q, const void *k, const void *v,
                                   const void *dout, const float *lse, void *dq, void *dk, void *dv, void *ws,
                                   cudaStream_t st) {
    const DbWs w = db_ws(d, true);
    char *base = static_cast<char *>(ws);
    DbArgs a = {};
    a.L = d.L; a.H = d.H; a.BH = d.B * d.H; a.ipc = 1; a.pos0 = pos0; a.scale = d.scale; a.dmax = dmax;
    a.Dx = Dx; a.delta = delta; a.hs_dx = hs_dx; a.hs_delta = hs_delta;
    a.lse = lse;
    a.ntab = (hs_dx != 0 || hs_delta != 0) ? d.H : 1;
    if (a.ntab > 1 && !d.periods) return cudaErrorInvalidValue;   // the tables are sized per head only then
    a.states = reinterpret_cast<__nv_bfloat16 *>(base + w.states);
    a.zbuf = reinterpret_cast<__nv_bfloat16 *>(base + w.z);
    a.etab = reinterpret_cast<uint8_t *>(base + w.etab);
    a.ctab = reinterpret_cast<uint8_t *>(base + w.ctab);
    a.err = device_error_word();
    if (d.dk == 64) return d.S == 32 ? launch_dbwd_t<64, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                                     : launch_dbwd_t<64, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
    return d.S == 32 ? launch_dbwd_t<128, 32>(d, a, q, k, v, dout, dq, dk, dv, st)
                     : launch_dbwd_t<128, 64>(d, a, q, k, v, dout, dq, dk, dv, st);
}

cudaError_t launch_decay_chunk(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                               int hs_dx, int hs_delta, const void *q, const void *k, const void *v, void *o,
                               float *lse, const float *state_in, float *state_out, void *ws, cudaStream_t st) {
    const DbWs w = db_ws(d, false);
    char *base = static_cast<char *>(ws);
    DbArgs a = {};
    a.L = d.L; a.H = d.H; a.BH = d.B * d.H; a.ipc = 1; a.pos0 = pos0; a.scale = d.scale; a.dmax = dmax;
    a.Dx = Dx; a.delta = delta; a.hs_dx = hs_dx; a.hs_delta = hs_delta;
    a.lse_out = lse;
    a.state_in = state_in;
    a.state_out = state_out;
    a.ntab = (hs_dx != 0 || hs_delta != 0) ? d.H : 1;
    if (a.ntab > 1 && !d.periods) return cudaErrorInvalidValue;   // the tables are sized per head only then
    a.states = reinterpret_cast<__nv_bfloat16 *>(base + w.states);
    a.etab = reinterpret_cast<uint8_t *>(base + w.etab);
    a.ctab = reinterpret_cast<uint8_t *>(base + w.ctab);
    a.err = device_error_word();
    if (d.dk == 64) return d.S == 32 ? launch_dfwd_t<64, 32>(d, a, q, k, v, o, st)
                                     : launch_dfwd_t<64, 64>(d, a, q, k, v, o, st);
    return d.S == 32 ? launch_dfwd_t<128, 32>(d, a, q, k, v, o, st) : launch_dfwd_t<128, 64>(d, a, q, k, v, o, st);
}

}  // namespace bla
