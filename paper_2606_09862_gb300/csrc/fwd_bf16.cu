// fwd_bf16.cu -- bf16 chunked forward on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Chunk algebra (the same exact rearrangement as the fp32 path, Eqs. (recurrence),
// (compressed), (output)), with the states kept in the absolute frame
// A_m = sum_{u < t0} e^{-i m w u} x_u (interleaved rows 2m = Re, 2m+1 = Im), for a chunk of
// C = 128 tokens starting at t0:
//   P  = tril(Q K^T)                                 [C x C]
//   X  = P EB_c^T + Q A^T,  EB_c[2m][u] = cos(m w (t0+u)), EB_c[2m+1][u] = -sin(m w (t0+u))
//   Y  = e^{i m w t} X (per row, t = t0 + row)       = q_t . Z_m(t)   (lag-frame state)
//   s  = scale Y PHI^T,   PHI[j][2m] = c_m cos(m w D_j), PHI[j][2m+1] = c_m sin(m w D_j)
//   p  = softmax over slots with t >= D_j
//   U  = p PHI;  A'  = rotation of U by -m w t  (real form of U_m e^{i m w t}, imaginary negated)
//   G  = tril(A' EB_c),  O = G V + A' A_V
//   A <- A + EB_c X_chunk  for X in {K, V}   (no rotation between chunks)
// The absolute-phase form (Alg. 1) differs only in its read-out: Y = X and A' = U (no per-row
// rotation) with the sine half of PHI negated.  The state is the same in both forms.
//
// The work runs as five kernels per call:
//   k_tables_bf16  EB_c of every chunk, PHI, the segment phase table and the slot lags
//   k_prepass  per (head, segment): segment deltas  F_seg [K|V]  (one GEMM, K-dim = segment)
//   k_scan     per head: states entering each segment, W_in(g+1) = e^{i m w Lseg} W_in(g) + delta(g)
//   k_kpass    per (head, segment): carries the K state in TMEM, writes slot probabilities p and lse
//   k_vpass    per (head, segment): carries the V state in TMEM, reads p, writes o
// The prepass runs 6 warps: warps 0-3 drain TMEM (thread = TMEM lane), warp 4 issues TMA loads,
// warp 5 allocates TMEM and issues the MMAs.  All waits are bounded (tc::mbar_wait).
#include <math.h>

#include "fwd_bf16.cuh"
#include "tc.cuh"
#include "tmap.cuh"

namespace bla {

namespace {

using bf16 = __nv_bfloat16;
constexpr int kC = 128;          // tokens per chunk (MMA M)
constexpr int kThreads = 192;
// The K and V passes run 12 warps: 0-7 drain TMEM as two warpgroups that split every row's
// columns in halves (warp w reads TMEM lanes 32(w%4)..), 8 issues TMA loads, 9 issues the MMAs,
// 10 issues the bulk stores of finished output tiles (K pass), 11 only completes the third
// warpgroup.  In the K pass the third warpgroup hands registers to the first two: launched with
// kLaunchRegs each (65536 / 384 rounded down to the allocation granule), it drops to kCtlRegs and
// the epilogue warpgroups rise to kEpiRegs, within the launch's total.  At 88 the control warps do not
// spill (at 40 the MMA issuer did, which measured slower), and the epilogue's rolled drains fit in 208.
// (The V pass measured slower with the same split and keeps kLaunchRegs everywhere.)
constexpr int kPassThreads = 384;
constexpr int kLaunchRegs = 168, kCtlRegs = 88, kEpiRegs = 208;
static_assert(128 * kCtlRegs + 256 * kEpiRegs <= kPassThreads * kLaunchRegs, "register split exceeds the launch");
constexpr int kPassEpiWarps = 8;


// ------------------------------------------------------------------ geometry

struct Geo {
    int BH, L, D, M, R2, RH, NH, NB, S, SP, RP;
    int nchunks, cps, G, Lseg;      // chunks per segment, segments per head, segment length (tokens)
};

// Multiprocessors of the current device (queried once per device).
static int sm_count() {
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
        cached[dev] = n;
    }
    return cached[dev];
}

Geo make_geo(const OpDims &d) {
    Geo g;
    g.BH = d.B * d.H; g.L = d.L; g.D = d.dk; g.M = d.M; g.R2 = d.R2;
    g.RH = d.R2 < 128 ? d.R2 : 128;
    g.NH = d.R2 / g.RH;
    g.NB = d.R2 <= 128 ? 1 : d.R2 / 128;
    g.RP = g.NB * 128;
    g.S = d.S;
    g.SP = d.S < 64 ? 64 : d.S;
    g.nchunks = (d.L + kC - 1) / kC;
    // Segments per head.  The passes run one CTA per SM; a CTA costs about (chunks + 2) chunk
    // periods (state entry and pipeline fill come to ~2), both passes run on the same grid, and
    // with more than one segment the prepass adds ~0.3 chunk period per chunk.  Pick the count
    // that minimises waves x that cost.
    const int nsm = sm_count();
    g.cps = g.nchunks > 0 ? g.nchunks : 1;
    double best = 1e300;
    for (int G = 1; G <= g.nchunks && G <= 256; ++G) {
        const int cps = (g.nchunks + G - 1) / G;
        const int Geff = (g.nchunks + cps - 1) / cps;
        if (Geff != G) continue;
        const long long waves = ((long long)g.BH * G + nsm - 1) / nsm;
        const double cost = (double)waves * (2.0 * (cps + 2) + (G > 1 ? 0.3 * cps : 0.0));
        if (cost < best - 1e-9) {
            best = cost;
            g.cps = cps;
        }
    }
    g.G = g.nchunks > 0 ? (g.nchunks + g.cps - 1) / g.cps : 1;
    g.Lseg = g.cps * kC;
    return g;
}

struct WsLayout {
    size_t delta, eb, phi, fseg, hw, htint, deltas, win, pbuf, total;
};

// With per-head periods every table is repeated per head (nh = H), plus each head's mode frequency
// and integer period; with one shared period nh = 1 and the head arrays are absent.
WsLayout ws_layout(const OpDims &d, const Geo &g) {
    WsLayout w;
    const size_t nh = d.periods ? (size_t)d.H : 1;
    size_t off = 0;
    w.delta = off;  off += align_up(sizeof(int) * nh * g.S, 1024);
    w.eb = off;     off += align_up(sizeof(bf16) * nh * g.nchunks * g.RP * kC, 1024);   // EB per chunk
    w.phi = off;    off += align_up(sizeof(bf16) * nh * g.SP * g.R2, 1024);
    w.fseg = off;   off += g.G > 1 ? align_up(sizeof(bf16) * nh * g.RP * g.Lseg, 1024) : 0;
    w.hw = off;     off += d.periods ? align_up(sizeof(double) * nh, 256) : 0;
    w.htint = off;  off += d.periods ? align_up(sizeof(int) * nh, 256) : 0;
    w.deltas = off; off += g.G > 1 ? align_up(sizeof(float) * (size_t)g.BH * g.G * 2 * g.RP * g.D, 1024) : 0;
    w.win = off;    off += g.G > 1 ? align_up(sizeof(float) * (size_t)g.BH * g.G * 2 * g.RP * g.D, 1024) : 0;
    w.pbuf = off;   off += align_up(sizeof(bf16) * (size_t)g.BH * (g.L > 0 ? g.L : 1) * g.SP, 1024);
    w.total = off;
    return w;
}

// ------------------------------------------------------------------ bf16 tables

// (cos, sin)(m w u): with w = 2 pi / T and an integer period tint > 0 the angle is reduced
// exactly, 2 pi ((m u) mod T) / T, and evaluated by sincospi in fp32; otherwise in fp64.
__device__ __forceinline__ void mode_phase(long long mu, double w, int tint, float *c, float *s) {
    if (tint > 0) {
        const int kk = mu < 0x7fffffffLL ? (int)((unsigned)mu % (unsigned)tint) : (int)(mu % tint);
        sincospif(2.0f * (float)kk / (float)tint, s, c);
    } else {
        double sd, cd;
        sincos((double)mu * w, &sd, &cd);
        *s = (float)sd;
        *c = (float)cd;
    }
}

// Operand tables of the tensor-core path, in bf16 (rows beyond 2M and slots beyond S are zero):
//   EB    [nch][RP][C]: EB_c[2m][u] = cos(m w (cC + u)), EB_c[2m+1][u] = -sin(m w (cC + u));
//         with nch = 1 this is the in-chunk table (c = 0) of the lag frame
//   PHI   [SP][R2]: PHI[j][2m] = c_m cos(m w D_j), PHI[j][2m+1] = sigma c_m sin(m w D_j), D_j = round(j T / S),
//         c_0 = 1/(2M-1), c_m = 2/(2M-1); sigma = +1 (lag form) or -1 (absolute form, Alg. 1)
//   FSEG  [RP][Lseg] (optional): FSEG[2m][u] = cos(m w (Lseg - u)), FSEG[2m+1][u] = sin(m w (Lseg - u)),
//         eight entries per thread as for EB
//   delta [S] (optional): the slot lags D_j
// EB is written by one thread per (c, m, 8 consecutive u), u fastest so that a warp writes whole
// rows: the first phase is reduced exactly, the next seven follow by products with e^{i m w}.
// Per-head periods (Alg. 1 and Alg. 3: T in R^H; hp.n = H > 0): head h writes its own copy of every
// table at (T_h, w_h, tint_h), one table block after the other, and hw[h], htint[h]; with hp.n = 0
// the single (T, w, tint) is used.
struct HeadTint {
    int t[kMaxHeadPeriods];   // each head's integer period for exact phase reduction (0: fp64 phases)
};

// One EB item of one head's table `eb` ([nch][RP][C]): rows 2m and 2m+1 of chunk c for 8 consecutive u,
// item ui = (c MP + m) (C / 8) + u0 / 8 (u fastest, so that a warp writes whole rows).
__device__ __forceinline__ void eb_item(bf16 *eb, int M, int RP, unsigned ui, double w, int tint) {
    // (32-bit index arithmetic: nch MP C / 8 = 16 L < 2^31 for L <= 2^26, which the host checks)
    const unsigned per_c = (unsigned)(RP / 2) * (kC / 8);
    const int c = (int)(ui / per_c), rem = (int)(ui - (unsigned)c * per_c);
    const int m = rem / (kC / 8), u0 = (rem % (kC / 8)) * 8;
    bf16 *rc = eb + ((size_t)c * RP + 2 * m) * kC + u0, *rs = rc + kC;
    uint32_t wc[4] = {0u, 0u, 0u, 0u}, ws[4] = {0u, 0u, 0u, 0u};
    if (m < M) {
        float bc, bs, ec, es;
        mode_phase((long long)m * ((long long)c * kC + u0), w, tint, &bc, &bs);
        mode_phase((long long)m, w, tint, &ec, &es);
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
            const float c0 = bc, s0 = bs;
            float t = bc * ec - bs * es;
            bs = bc * es + bs * ec;
            bc = t;
            wc[j / 2] = tc::pack_bf16x2(c0, bc);
            ws[j / 2] = tc::pack_bf16x2(-s0, -bs);
            t = bc * ec - bs * es;
            bs = bc * es + bs * ec;
            bc = t;
        }
    }
    *reinterpret_cast<uint4 *>(rc) = make_uint4(wc[0], wc[1], wc[2], wc[3]);
    *reinterpret_cast<uint4 *>(rs) = make_uint4(ws[0], ws[1], ws[2], ws[3]);
}

// With eb_skip the EB tables are left to the segment prepass (whose epilogue warps are idle while
// its MMAs stream K and V); everything else is written here.
__global__ void k_tables_bf16(int M, int S, int SP, int RP, int Lseg, int nch, HeadPeriods hp, HeadTint ht, double T0,
                              double w0, int tint0, float sin_sign, bf16 *eb0, bf16 *phi0, bf16 *fseg0, int *delta0,
                              double *hw, int *htint, int eb_skip) {
    const int R2 = 2 * M, MP = RP / 2;
    const long long n_eb = eb_skip ? 0 : (long long)nch * MP * (kC / 8), n_phi = (long long)SP * R2;
    const long long n_f = fseg0 ? (long long)MP * ((Lseg + 7) / 8) : 0, n_d = delta0 ? S : 0;
    const long long per = n_eb + n_phi + n_f + n_d + 1;
    const int nh = hp.n > 0 ? hp.n : 1;
    const long long total = per * nh;
    const double n = 2.0 * M - 1.0;
    for (long long ii = blockIdx.x * (long long)blockDim.x + threadIdx.x; ii < total;
         ii += (long long)gridDim.x * blockDim.x) {
        const int h = hp.n > 0 ? (int)(ii / per) : 0;   // (one shared period: ii < per)
        const long long i = ii - (long long)h * per;
        const double T = hp.n > 0 ? hp.T[h] : T0, w = hp.n > 0 ? hp.w[h] : w0;
        const int tint = hp.n > 0 ? ht.t[h] : tint0;
        bf16 *eb = eb0 + (size_t)h * nch * RP * kC, *phi = phi0 + (size_t)h * SP * R2;
        bf16 *fseg = fseg0 ? fseg0 + (size_t)h * RP * Lseg : nullptr;
        int *delta = delta0 ? delta0 + (size_t)h * S : nullptr;
        if (i == per - 1) {
            if (hp.n > 0) {
                hw[h] = w;
                htint[h] = tint;
            }
        } else if (i < n_eb) {
            eb_item(eb, M, RP, (unsigned)i, w, tint);
        } else if (i < n_eb + n_phi) {
            const int e = (int)(i - n_eb);
            const int j = e / R2, r = e % R2, m = r >> 1;
            float v = 0.f;
            if (j < S) {
                const long long dj = (long long)rint((double)j * T / (double)S);
                const float cm = (m == 0) ? (float)(1.0 / n) : (float)(2.0 / n);
                float c, sn;
                mode_phase((long long)m * dj, w, tint, &c, &sn);
                v = cm * ((r & 1) ? sin_sign * sn : c);
            }
            phi[e] = __float2bfloat16_rn(v);
        } else if (i < n_eb + n_phi + n_f) {
            // FSEG rows 2m, 2m+1 for 8 consecutive u: e^{i m w (Lseg - u)}, stepping by e^{-i m w}
            const int e = (int)(i - n_eb - n_phi);
            const int per_m = (Lseg + 7) / 8;
            const int m = e / per_m, u0 = (e % per_m) * 8;
            bf16 *rc = fseg + (size_t)(2 * m) * Lseg + u0, *rs = rc + Lseg;
            float bc = 0.f, bs = 0.f, ec = 1.f, es = 0.f;
            if (m < M) {
                mode_phase((long long)m * (Lseg - u0), w, tint, &bc, &bs);
                mode_phase((long long)m, w, tint, &ec, &es);
            }
            float vc[8], vs[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                vc[j] = bc;
                vs[j] = bs;
                const float t = bc * ec + bs * es;   // times e^{-i m w}
                bs = bs * ec - bc * es;
                bc = t;
            }
            if (u0 + 8 <= Lseg && (Lseg & 7) == 0) {   // whole 16-byte pieces of 16-byte aligned rows
                *reinterpret_cast<uint4 *>(rc) = make_uint4(tc::pack_bf16x2(vc[0], vc[1]), tc::pack_bf16x2(vc[2], vc[3]),
                                                            tc::pack_bf16x2(vc[4], vc[5]), tc::pack_bf16x2(vc[6], vc[7]));
                *reinterpret_cast<uint4 *>(rs) = make_uint4(tc::pack_bf16x2(vs[0], vs[1]), tc::pack_bf16x2(vs[2], vs[3]),
                                                            tc::pack_bf16x2(vs[4], vs[5]), tc::pack_bf16x2(vs[6], vs[7]));
            } else {
                for (int j = 0; j < 8 && u0 + j < Lseg; ++j) {
                    rc[j] = __float2bfloat16_rn(vc[j]);
                    rs[j] = __float2bfloat16_rn(vs[j]);
                }
            }
        } else {
            const int j = (int)(i - n_eb - n_phi - n_f);
            delta[j] = (int)rint((double)j * T / (double)S);
        }
    }
}

// ------------------------------------------------------------------ kernel arguments

struct Args {
    Geo g;
    float scale;
    double w;
    const int *delta;    // [S]
    const float *deltas; // [BH][G][2][RP][D] segment deltas (prepass output)
    float *win;          // [BH][G][2][RP][D] states entering each segment (or null if G == 1)
    bf16 *pbuf;          // [BH][L][SP]
    float *lse;          // [BH][L] or null
    bf16 *o;             // [BH][L][D]
    float *state_out;    // [BH][2][M][2][D] or null
    float *deltas_out;   // prepass output (same buffer as deltas)
    int tint;            // integer period for exact phase reduction (0: use fp64 phases)
    int absolute;        // absolute form (Alg. 1): the drains do not rotate rows by e^{i m w t}
    int *err;
    // Per-head periods (Alg. 1 and Alg. 3: T in R^H): head h = bh % H reads its own tables at these
    // per-head strides (rows of the EB, PHI and FSEG tensor maps; entries of delta) and its own w and
    // integer period; all four strides are 0 and hw, htint null when the heads share one period.
    int H;
    int eb_rows_h, phi_rows_h, f_rows_h, delta_h;
    const double *hw;
    const int *htint;
    // EB tables written by the prepass's epilogue warps while its MMAs run (null: the tables kernel
    // wrote them); eb_nh heads of [nchunks][RP][C] each
    bf16 *eb_gen;
    int eb_nh;
};

// Mode frequency and integer period of head bh % H (written by the tables kernel: read them only
// after the programmatic-launch wait).
struct HeadW {
    double w;
    int tint;
};
__device__ __forceinline__ HeadW head_w(const Args &a, int bh) {
    if (!a.hw) return HeadW{a.w, a.tint};
    const int hd = bh % a.H;
    return HeadW{a.hw[hd], a.htint[hd]};
}

// Bounded-wait bookkeeping shared by the roles of one CTA.
struct Ctl {
    volatile int abort;
    int kernel;            // 1 prepass, 2 K pass, 3 V pass
    uint64_t *bar0;        // first barrier of the CTA (for error reports)
};

// Bounded wait on `bar` for the phase of parity `phase` (flipped after the call).  On a
// timeout the CTA's abort flag is raised and the error word records
//   DEVERR_MBAR_TIMEOUT | kernel << 4 | barrier index << 8 | parity << 15 | block << 16.
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t &phase, Ctl *ctl, int *err) {
    if (ctl->abort) return false;
    bool ok = tc::mbar_wait(bar, phase);
    if (!ok) {
        ctl->abort = 1;
        report_device_error(err, DEVERR_MBAR_TIMEOUT | (ctl->kernel << 4) |
                                     ((int)(bar - ctl->bar0) << 8) | ((int)phase << 15) | ((int)blockIdx.x << 16));
    }
    phase ^= 1u;
    return ok;
}

// wait_bar on the parity stored in bit `bit` of `bits` (flipped afterwards).
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t &bits, int bit, Ctl *ctl, int *err) {
    uint32_t ph = (bits >> bit) & 1u;
    const bool ok = wait_bar(bar, ph, ctl, err);
    bits ^= 1u << bit;
    return ok;
}

// Epilogue hand-off: every thread has finished its TMEM reads/writes and shared-memory
// stores (fenced by the caller); the warp converges and its lane 0 arrives once.
__device__ __forceinline__ void epi_arrive(uint64_t *bar) {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) tc::mbar_arrive(bar);
}

// Bounded barrier among the epilogue warps (an mbarrier counting one arrival per warp):
// every epilogue thread arrives through its warp and waits for the phase to complete.
__device__ __forceinline__ bool epi_sync(uint64_t *bar, uint32_t &phase, Ctl *ctl, int *err) {
    epi_arrive(bar);
    return wait_bar(bar, phase, ctl, err);
}

__device__ __forceinline__ uint32_t tmem_addr(uint32_t base, int lane_base, int col) {
    return base + ((uint32_t)lane_base << 16) + (uint32_t)col;
}

// Store 32 fp32 values of one tile row as bf16 into a [rows][64]-blocked 128B-swizzled tile,
// columns [col0, col0+32) (col0 a multiple of 32).
__device__ __forceinline__ void st_row32_bf16(uint8_t *tile, int rows_per_block, int row, int col0, const float *v) {
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

// MMA helpers: one K-step of 16 on 128B-swizzled tiles.
//   K-major tile: blocks of [rows][64] (block bytes = rows*128); step k -> block k/4, +32B*(k%4).
__device__ __forceinline__ uint64_t kmaj_desc(const uint8_t *tile, int rows, int k) {
    uint32_t a = tc::smem_u32(tile) + (uint32_t)((k >> 2) * rows * 128) + (uint32_t)((k & 3) * 32);
    return tc::sdesc_sw128(a, 16, 1024);
}
//   MN-major tile: [K rows][64 MN] blocks, block bytes = krows*128 (LBO); step k -> +16 rows.
__device__ __forceinline__ uint64_t mnmaj_desc(const uint8_t *tile, int krows, int k) {
    uint32_t a = tc::smem_u32(tile) + (uint32_t)(k * 16 * 128);
    return tc::sdesc_sw128(a, (uint32_t)krows * 128u, 1024);
}

// (cos, sin)(m w t) for the product mt = m t, reduced exactly when w = 2 pi / tint.
__device__ __forceinline__ float2 abs_phase(long long mt, double w, int tint) {
    float c, s;
    mode_phase(mt, w, tint, &c, &s);
    return make_float2(c, s);
}

__device__ __forceinline__ float2 cmul(float2 a, float2 b) {
    return make_float2(a.x * b.x - a.y * b.y, a.x * b.y + a.y * b.x);
}

// Phases of token t for the drains of one chunk: e^{i m0 w t} for the first mode of this thread's
// range in each half (h0, h1), e^{i w t} (start offset of the second interleaved chain) and
// e^{i 2 w t} (step of both chains).
struct RowPhases {
    float2 e1, e2, h0, h1;
};
__device__ __forceinline__ RowPhases row_phases(long long t, int m00, int m10, bool two, double w, int tint) {
    RowPhases p;
    p.e1 = abs_phase(t, w, tint);
    p.e2 = abs_phase(2 * t, w, tint);
    p.h0 = abs_phase((long long)m00 * t, w, tint);
    p.h1 = two ? abs_phase((long long)m10 * t, w, tint) : make_float2(1.f, 0.f);
    return p;
}
// The phases of token t + C from those of t and the phases of C (one complex product each; over
// the chunks of one segment the rounding stays orders of magnitude below bf16 resolution).
__device__ __forceinline__ void advance(RowPhases &p, const RowPhases &step) {
    p.e1 = cmul(p.e1, step.e1);
    p.e2 = cmul(p.e2, step.e2);
    p.h0 = cmul(p.h0, step.h0);
    p.h1 = cmul(p.h1, step.h1);
}

// Initial state block in the absolute frame: the carried-in lag-frame state S (rows [rows][stride],
// interleaved (Re, Im) row pairs; null = zero) rotated to A = e^{-i m w t0} S, written to TMEM.
// (c, s) = (cos, sin)(m w t0) of this thread's mode.  Each thread loads only its own row, all
// loads issued before any use (one memory latency per block); the partner row of the pair is
// the neighbouring lane's.
// L2 prefetch of this thread's DH columns of one state row (issued before an earlier block is
// processed, so that the later block's loads do not pay the full memory latency).
template <int DH>
__device__ __forceinline__ void state_prefetch_row(const float *src, int row, int live_rows, int stride) {
    if (src == nullptr || row >= live_rows) return;
    const float *p = src + (size_t)row * stride;
#pragma unroll
    for (int i = 0; i < DH; i += 32) asm volatile("prefetch.global.L2 [%0];" ::"l"(p + i) : "memory");
}

template <int DH>
__device__ __forceinline__ void state_init_abs(uint32_t tbase, int col0, int row, const float *src, int live_rows,
                                               int stride, float c, float s) {
    const int lane_base = (row >> 5) << 5;
    const float sg = (row & 1) ? -s : s;   // Re' = c Re + s Im ; Im' = c Im - s Re
    const bool live = src != nullptr && row < live_rows;   // same for both rows of a pair
    float v[DH];
#pragma unroll
    for (int i = 0; i < DH; i += 4) {
        float4 t = make_float4(0.f, 0.f, 0.f, 0.f);
        if (live) t = __ldg(reinterpret_cast<const float4 *>(src + (size_t)row * stride + i));
        v[i] = t.x;
        v[i + 1] = t.y;
        v[i + 2] = t.z;
        v[i + 3] = t.w;
    }
#pragma unroll
    for (int i = 0; i < DH; ++i) {
        const float par = __shfl_xor_sync(0xffffffffu, v[i], 1);
        v[i] = c * v[i] + sg * par;
    }
    tc::tmem_st<DH>(tmem_addr(tbase, lane_base, col0), v);
}

// Load DH columns of this thread's state row from TMEM and pack them to bf16 pairs.
template <int DH>
__device__ __forceinline__ void state_pack(uint32_t tbase, int col0, int row, uint32_t *pk) {
    const int lane_base = (row >> 5) << 5;
#pragma unroll
    for (int p0 = 0; p0 < DH; p0 += 32) {
        float v[32];
        tc::tmem_ld<32>(tmem_addr(tbase, lane_base, col0 + p0), v);
#pragma unroll
        for (int i = 0; i < 32; i += 2) pk[(p0 + i) / 2] = tc::pack_bf16x2(v[i], v[i + 1]);
    }
}

// Store 32 bf16 values (16 packed words) of one tile row, like st_row32_bf16.
__device__ __forceinline__ void st_row32_packed(uint8_t *tile, int rows_per_block, int row, int col0,
                                                const uint32_t *pk) {
    uint8_t *blk = tile + (size_t)(col0 >> 6) * rows_per_block * 128;
    const int c = col0 & 63;
#pragma unroll
    for (int q = 0; q < 4; ++q)
        *reinterpret_cast<uint4 *>(blk + tc::sw128_offset(row, c + q * 8)) =
            make_uint4(pk[q * 4 + 0], pk[q * 4 + 1], pk[q * 4 + 2], pk[q * 4 + 3]);
}

// Descriptor offset of K-step k from step 0, in the 16-byte units of the address field (tiles
// lie below 256 KiB, so the sum never carries out of the field).
__device__ __forceinline__ uint64_t kmaj_step(int rows, int k) {
    return (uint64_t)((((k >> 2) * rows * 128) + (k & 3) * 32) >> 4);
}
__device__ __forceinline__ uint64_t mnmaj_step(int k) { return (uint64_t)(k * 128); }   // 16 rows x 128 B

// An opaque copy of x: values derived from it cannot be hoisted above this point.
__device__ __forceinline__ uint64_t opaque(uint64_t x) {
    asm volatile("" : "+l"(x));
    return x;
}

// acc (+)= A B^T over nk K-steps of 16.  A is a K-major tile of `arows` rows; B is K-major with
// `brows` rows, or MN-major (MN_B) with `brows` K rows per block.  The first step accumulates only
// if acc0.  Each step's descriptors are the base descriptors plus a constant, formed at the issue,
// so that the issuing thread holds two descriptors rather than one per step.
template <bool MN_B>
__device__ __forceinline__ void mma_steps(uint32_t acc, const uint8_t *a, int arows, const uint8_t *b, int brows,
                                          uint32_t idesc, int nk, bool acc0) {
    const uint64_t da = opaque(kmaj_desc(a, arows, 0));
    const uint64_t db = opaque(MN_B ? mnmaj_desc(b, brows, 0) : kmaj_desc(b, brows, 0));
#pragma unroll
    for (int k = 0; k < nk; ++k)
        tc::mma_bf16(acc, da + kmaj_step(arows, k), db + (MN_B ? mnmaj_step(k) : kmaj_step(brows, k)), idesc,
                     (acc0 || k > 0) ? 1u : 0u);
}

// Rotate the state block held in TMEM (rows = lanes, interleaved cos/sin pairs) by the
// phase (c, s) of this thread's mode, optionally write it back, and emit a bf16 copy into
// a [RH rows][64 d]-blocked tile (rows >= RH skipped) and/or an fp32 copy to global.
// Executed by the 128 epilogue threads; `row` is this thread's lane = local state row.
template <int D>
__device__ __forceinline__ void state_pass(uint32_t tbase, int col0, int row, bool rotate, float c, float s,
                                           bool write_back, uint8_t *wtile, int RH, float *gout, int ccol = 0) {
    const int lane_base = (row >> 5) << 5;
    const uint32_t addr = tmem_addr(tbase, lane_base, col0);
    float v[D];
    tc::tmem_ld<D>(addr, v);
    if (rotate) {
        const bool odd = row & 1;
#pragma unroll
        for (int i = 0; i < D; ++i) {
            const float partner = __shfl_xor_sync(0xffffffffu, v[i], 1);
            // even row: Re' = c Re - s Im ; odd row: Im' = s Re + c Im
            v[i] = odd ? fmaf(s, partner, c * v[i]) : fmaf(-s, partner, c * v[i]);
        }
        if (write_back) tc::tmem_st<D>(addr, v);
    }
    if (wtile && row < RH) {
#pragma unroll
        for (int g = 0; g < D; g += 32) st_row32_bf16(wtile, RH, row, ccol + g, v + g);
    }
    if (gout) {
#pragma unroll
        for (int i = 0; i < D; i += 4)
            *reinterpret_cast<float4 *>(gout + ccol + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
}

// ================================================================== prepass
//
// delta_seg[K|V][RP][D] = F_seg [RP x Lseg] . X_seg [Lseg x D] for every full segment but the last.
// Pipelined over half-chunks of 64 tokens with 3 smem stages.

constexpr int kPreStages = 3;

__global__ void __launch_bounds__(kThreads, 1)
    k_prepass(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
              const __grid_constant__ CUtensorMap tm_f, const __grid_constant__ CUtensorMap tm_d, Args a) {
    const Geo &g = a.g;
    const int seg = blockIdx.x % g.G, bh = blockIdx.x / g.G;
    if (seg >= g.G - 1) return;   // the last segment's delta is never used
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int D = g.D, NB = g.NB;
    const size_t f_bytes = (size_t)NB * 128 * 64 * 2, x_bytes = (size_t)64 * D * 2;
    const size_t stage_bytes = f_bytes + 2 * x_bytes;
    uint8_t *stage0 = sm;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + kPreStages * stage_bytes);
    uint64_t *full = bars, *empty = bars + kPreStages, *done = bars + 2 * kPreStages;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 2 * kPreStages + 1);
    Ctl *ctl = reinterpret_cast<Ctl *>(bars + 2 * kPreStages + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t ncols = (uint32_t)(2 * NB * D) <= 128 ? 128u : (uint32_t)(2 * NB * D) <= 256 ? 256u : 512u;
    // (the host requests shared memory so that CTAs whose column counts would not fit together
    //  are never co-resident)

    if (threadIdx.x == 0) {
        for (int i = 0; i < kPreStages; ++i) { tc::mbar_init(&full[i], 1); tc::mbar_init(&empty[i], 1); }
        tc::mbar_init(done, 1);
        ctl->abort = 0;
        ctl->kernel = 1;
        ctl->bar0 = bars;
        tc::fence_barrier_init();
    }
    if (warp == 5) { tc::tmem_alloc(tslot, ncols); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;
    tc::pdl_wait();      // the tables
    const int steps = g.cps * 2;          // half-chunks in the segment
    const int t_seg = seg * g.Lseg;

    if (warp == 4 && lane == 0) {
        const int fy = (bh % a.H) * a.f_rows_h;   // this head's FSEG rows
        uint32_t ph[kPreStages] = {0, 0, 0};
        for (int it = 0; it < steps; ++it) {
            const int st = it % kPreStages;
            if (it >= kPreStages && !wait_bar(&empty[st], ph[st], ctl, a.err)) break;
            uint8_t *base = stage0 + st * stage_bytes;
            tc::mbar_arrive_expect_tx(&full[st], (uint32_t)stage_bytes);
            for (int b = 0; b < NB; ++b)
                tc::tma_load_2d(base + b * 128 * 128, &tm_f, &full[st], it * 64, fy + b * 128);
            for (int db = 0; db < D / 64; ++db) {
                tc::tma_load_3d(base + f_bytes + db * 64 * 128, &tm_k, &full[st], db * 64, t_seg + it * 64, bh);
                tc::tma_load_3d(base + f_bytes + x_bytes + db * 64 * 128, &tm_v, &full[st], db * 64, t_seg + it * 64,
                                bh);
            }
        }
    } else if (warp == 5 && lane == 0) {
        uint32_t ph[kPreStages] = {0, 0, 0};
        // K and V of a stage are adjacent MN-major blocks of [64 tokens][64 d] (LBO = 8 KB), so one
        // N = 2D MMA covers both: accumulator columns [b*2D, b*2D + D) for K, [b*2D + D, (b+1)*2D) for V
        const uint32_t idesc = tc::idesc_bf16(128, 2 * D, false, true);
        for (int it = 0; it < steps; ++it) {
            const int st = it % kPreStages;
            if (!wait_bar(&full[st], ph[st], ctl, a.err)) break;
            tc::tc_fence_after();
            uint8_t *base = stage0 + st * stage_bytes;
            for (int b = 0; b < NB; ++b)
                for (int k = 0; k < 4; ++k) {
                    uint64_t ad = kmaj_desc(base + b * 128 * 128, 128, k);
                    uint64_t bd = mnmaj_desc(base + f_bytes, 64, k);
                    tc::mma_bf16(tb + (uint32_t)(b * 2 * D), ad, bd, idesc, (it > 0 || k > 0) ? 1u : 0u);
                }
            tc::mma_commit(&empty[st]);
        }
        tc::mma_commit(done);
    } else if (warp < 4) {
        if (a.eb_gen) {
            // this CTA's share of the EB tables (the CTAs of every segment but the last get here)
            const unsigned n_eb = (unsigned)g.nchunks * (unsigned)(g.RP / 2) * (kC / 8);
            const unsigned nct = (unsigned)g.BH * (unsigned)(g.G - 1), ci = (unsigned)bh * (g.G - 1) + seg;
            const unsigned nitems = n_eb * (unsigned)a.eb_nh;
            for (unsigned i = ci * 128u + threadIdx.x; i < nitems; i += nct * 128u) {
                const int h = (int)(i / n_eb);
                const double w = a.hw ? a.hw[h] : a.w;
                const int tint = a.hw ? a.htint[h] : a.tint;
                eb_item(a.eb_gen + (size_t)h * g.nchunks * g.RP * kC, g.M, g.RP, i - (unsigned)h * n_eb, w, tint);
            }
        }
        uint32_t ph = 0;
        bool ok = wait_bar(done, ph, ctl, a.err);
        tc::tc_fence_after();
        if (ok) {
            // The deltas leave through the (now idle) pipeline stages: thread = state row writes its
            // row into [NB][D/32][128 rows][32] fp32 boxes (128-byte swizzled), and thread 0 stores
            // them by TMA, K first, then V
            const int row = threadIdx.x, lane_base = (row >> 5) << 5;
            for (int x = 0; x < 2; ++x) {
                if (x > 0) {
                    if (row == 0) tc::bulk_wait_read0();   // the K boxes have been read
                    tc::named_bar(1, 128);
                }
                for (int b = 0; b < NB; ++b)
                    for (int cb = 0; cb < D / 32; ++cb) {
                        float v[32];
                        tc::tmem_ld<32>(tmem_addr(tb, lane_base, (b * 2 + x) * D + cb * 32), v);
                        uint8_t *box = stage0 + (size_t)(b * (D / 32) + cb) * 128 * 128;
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            *reinterpret_cast<float4 *>(box + row * 128 + ((q ^ (row & 7)) << 4)) =
                                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                    }
                tc::fence_proxy_async_smem();
                tc::named_bar(1, 128);
                if (row == 0) {
                    const int r0 = (int)((((size_t)bh * g.G + seg) * 2 + x) * g.RP);
                    for (int b = 0; b < NB; ++b)
                        for (int cb = 0; cb < D / 32; ++cb)
                            tc::tma_store_2d(&tm_d, stage0 + (size_t)(b * (D / 32) + cb) * 128 * 128, cb * 32,
                                             r0 + b * 128);
                    tc::bulk_commit();
                }
            }
            if (row == 0) tc::bulk_wait0();
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 5) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, ncols);
    }
}

// ================================================================== segment scan
// W_in(0) = 0; W_in(g+1) = e^{i m w Lseg} W_in(g) + delta(g).  One thread per (head, K|V, mode, four
// consecutive state columns): the index arithmetic and the mode's phase are paid once per four
// columns, and every access is 16 bytes wide.
__global__ void k_scan(Args a) {
    tc::pdl_wait();      // the segment deltas
    const Geo &g = a.g;
    const int vsh = g.D == 128 ? 5 : 4;   // float4 per state row: D / 4 = 32 or 16
    // (the host checks that the thread count fits 32 bits)
    const unsigned total = ((unsigned)g.BH * 2u * (unsigned)g.M) << vsh, uM = (unsigned)g.M;
    for (unsigned i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const int e = (int)(i & ((1u << vsh) - 1u)) * 4;
        unsigned r = i >> vsh;
        const int m = (int)(r % uM);
        r /= uM;
        const int x = (int)(r & 1u);
        const int bh = (int)(r >> 1);
        float c, s;
        const HeadW hw = head_w(a, bh);
        mode_phase((long long)m * g.Lseg, hw.w, hw.tint, &c, &s);
        float4 re = make_float4(0.f, 0.f, 0.f, 0.f), im = re;
        // rows 2m (Re) and 2m+1 (Im) of segment seg: base + seg * seg_stride
        const size_t seg_stride = (size_t)2 * g.RP * g.D;
        const size_t base = (((size_t)bh * g.G * 2 + x) * g.RP + 2 * m) * g.D + e;
        // the deltas of eight segments are loaded before they are used, so that their latencies overlap
        for (int s0 = 0; s0 < g.G; s0 += 8) {
            float4 dre[8], dim[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int seg = s0 + j;
                dre[j] = dim[j] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (seg + 1 < g.G) {
                    dre[j] = *reinterpret_cast<const float4 *>(a.deltas + base + seg * seg_stride);
                    dim[j] = *reinterpret_cast<const float4 *>(a.deltas + base + seg * seg_stride + g.D);
                }
            }
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int seg = s0 + j;
                if (seg >= g.G) break;
                *reinterpret_cast<float4 *>(a.win + base + seg * seg_stride) = re;
                *reinterpret_cast<float4 *>(a.win + base + seg * seg_stride + g.D) = im;
                const float4 nre = make_float4(c * re.x - s * im.x + dre[j].x, c * re.y - s * im.y + dre[j].y,
                                               c * re.z - s * im.z + dre[j].z, c * re.w - s * im.w + dre[j].w);
                const float4 nim = make_float4(s * re.x + c * im.x + dim[j].x, s * re.y + c * im.y + dim[j].y,
                                               s * re.z + c * im.z + dim[j].z, s * re.w + c * im.w + dim[j].w);
                re = nre;
                im = nim;
            }
        }
    }
}

// Packed fp32 pairs (f32x2): one instruction for two elementwise operations, each rounded as the scalar
// operation would be.  The softmax uses them for its scale, exponent argument, sums and normalisation,
// which shortens the epilogue's instruction stream per chunk.
__device__ __forceinline__ void mul2_bcast(float &x, float &y, float s) {
    asm("{\n\t.reg .b64 a, b;\n\tmov.b64 a, {%0, %1};\n\tmov.b64 b, {%2, %2};\n\tmul.rn.f32x2 a, a, b;\n\t"
        "mov.b64 {%0, %1}, a;\n\t}"
        : "+f"(x), "+f"(y)
        : "f"(s));
}
__device__ __forceinline__ float2 sub2_bcast(float x, float y, float s) {
    float2 r;
    asm("{\n\t.reg .b64 a, b;\n\tmov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %4};\n\tsub.rn.f32x2 a, a, b;\n\t"
        "mov.b64 {%0, %1}, a;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(x), "f"(y), "f"(s));
    return r;
}
__device__ __forceinline__ void add2(float &x, float &y, float a, float b) {
    asm("{\n\t.reg .b64 u, w;\n\tmov.b64 u, {%0, %1};\n\tmov.b64 w, {%2, %3};\n\tadd.rn.f32x2 u, u, w;\n\t"
        "mov.b64 {%0, %1}, u;\n\t}"
        : "+f"(x), "+f"(y)
        : "f"(a), "f"(b));
}

// ================================================================== K pass

struct KLayout {
    size_t q, k, p, w, y, eb, phi, bars, total;
};

__host__ __device__ inline KLayout k_layout(const Geo &g) {
    KLayout l;
    size_t off = 0;
    l.q = off;   off += (size_t)kC * g.D * 2;
    l.k = off;   off += (size_t)kC * g.D * 2;
    l.p = off;   off += (size_t)kC * kC * 2;
    l.w = off;   off += (size_t)g.RH * g.D * 2;
    l.y = off;   off += (size_t)kC * g.RH * 2;
    l.eb = off;  off += (size_t)128 * kC * 2;
    l.phi = off; off += (size_t)g.SP * g.RH * 2;
    l.bars = off; off += 3072;   // barriers, TMEM slot, control, slot lags [0, 1024); softmax exchange
    l.total = off;               // the dynamic shared memory base is 1024-aligned (checked by the kernel)
    return l;
}

// One barrier per use and per mode half: a barrier is never committed twice without the
// waiter's hand-back in between, so a parity wait can never fall two phases behind.
enum KBar {
    KB_QK_FULL, KB_QK_FREE, KB_EB_FULL, KB_EB_FREE, KB_PHI_FULL, KB_PHI_FREE,
    KB_ACC_FULL_A, KB_ACC_FULL_B, KB_ACC_FREE_A, KB_ACC_FREE_B,
    KB_P_READY, KB_W_READY, KB_W_FREE, KB_STATE_DONE, KB_STATE_DONE1, KB_Y_READY, KB_Y_FREE, KB_EPI_SYNC, KB_Y_STORED,
    KB_P_SMEM, KB_EXIT, KB_COUNT
};

template <int D, int RH, int S, int NH>
__global__ void __launch_bounds__(kPassThreads, 1)
    k_kpass(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
            const __grid_constant__ CUtensorMap tm_eb, const __grid_constant__ CUtensorMap tm_phi,
            const __grid_constant__ CUtensorMap tm_p, Args a) {
    const Geo &g = a.g;
    // heads fastest: the CTAs of one segment run in the same wave and share its EB tables in L2
    const int bh = blockIdx.x % g.BH, seg = blockIdx.x / g.BH;
    const int c_begin = seg * g.cps, c_end = min(g.nchunks, c_begin + g.cps);
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // the 128-byte-swizzled tiles need a 1024-aligned base; the layout reserves no slack for it
    if (tc::smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) report_device_error(a.err, DEVERR_SMEM_ALIGN | (2 << 4) | ((int)blockIdx.x << 16));
        return;
    }
    uint8_t *sm = smem_raw;
    const KLayout lay = k_layout(g);
    uint8_t *sQ = sm + lay.q, *sK = sm + lay.k, *sP = sm + lay.p, *sW = sm + lay.w, *sY = sm + lay.y;
    uint8_t *sEB = sm + lay.eb, *sPHI = sm + lay.phi;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + lay.bars);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + KB_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + KB_COUNT + 1);
    int *sdelta = reinterpret_cast<int *>(bar + KB_COUNT + 4);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int SP = g.SP;
    // TMEM columns: [0, NB*D) state; accA at NB*D (128 cols); accB after it (RH cols).
    const int colA = g.NB * D, colB = colA + 128;
    const uint32_t ncols = (uint32_t)(colB + RH) <= 256 ? 256u : 512u;   // host: pow2_cols(NB*D + 128 + RH)

    if (threadIdx.x == 0) {
        for (int i = 0; i < KB_COUNT; ++i) {
            const bool epi = i == KB_P_READY || i == KB_W_READY || i == KB_Y_READY || i == KB_ACC_FREE_A ||
                             i == KB_ACC_FREE_B || i == KB_EPI_SYNC || i == KB_P_SMEM;
            tc::mbar_init(&bar[i], epi ? kPassEpiWarps : 1);
        }
        ctl->abort = 0;
        ctl->kernel = 2;
        ctl->bar0 = bar;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, ncols); tc::tmem_relinquish(); }
    // the tables and the entering states come from the kernels before this one
    tc::pdl_wait();
    for (int j = threadIdx.x; j < S; j += blockDim.x) sdelta[j] = a.delta[(bh % a.H) * a.delta_h + j];
    const HeadW hph = head_w(a, bh);                      // this head's w and integer period
    const int eby = (bh % a.H) * a.eb_rows_h, phy = (bh % a.H) * a.phi_rows_h;   // its table rows
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;

    if (warp >= 8) {
        tc::reg_dealloc<kCtlRegs>();
        if (warp == 8) {
            // ---------------- TMA producer: per chunk Q, K, then (EB_h, PHI_h) for each mode half, in
            // the order the MMA issuer consumes them
            if (lane == 0) {
                tc::tma_prefetch_desc(&tm_q); tc::tma_prefetch_desc(&tm_k);
                tc::tma_prefetch_desc(&tm_eb); tc::tma_prefetch_desc(&tm_phi);
                uint32_t ph_qk = 0, ph_eb = 0, ph_phi = 0;
                bool first_eb = true, first_phi = true;
                for (int c = c_begin; c < c_end && !ctl->abort; ++c) {
                    if (c > c_begin && !wait_bar(&bar[KB_QK_FREE], ph_qk, ctl, a.err)) break;
                    tc::mbar_arrive_expect_tx(&bar[KB_QK_FULL], (uint32_t)(2 * kC * D * 2));
                    for (int db = 0; db < D / 64; ++db) {
                        tc::tma_load_3d(sQ + db * kC * 128, &tm_q, &bar[KB_QK_FULL], db * 64, c * kC, bh);
                        tc::tma_load_3d(sK + db * kC * 128, &tm_k, &bar[KB_QK_FULL], db * 64, c * kC, bh);
                    }
                    // the next chunk's q and k into L2 now: their loads wait for this chunk's state_1
                    // update and would otherwise pay the full memory latency on the chunk's critical path
                    if (c + 1 < c_end) {
                        for (int db = 0; db < D / 64; ++db) {
                            tc::tma_prefetch_3d(&tm_q, db * 64, (c + 1) * kC, bh);
                            tc::tma_prefetch_3d(&tm_k, db * 64, (c + 1) * kC, bh);
                        }
                    }
                    for (int h = 0; h < NH; ++h) {
                        if (!first_eb && !wait_bar(&bar[KB_EB_FREE], ph_eb, ctl, a.err)) break;
                        first_eb = false;
                        tc::mbar_arrive_expect_tx(&bar[KB_EB_FULL], (uint32_t)(128 * kC * 2));
                        for (int kb = 0; kb < 2; ++kb)
                            tc::tma_load_2d(sEB + kb * 128 * 128, &tm_eb, &bar[KB_EB_FULL], kb * 64,
                                            eby + c * g.RP + h * 128);
                        if (!first_phi && !wait_bar(&bar[KB_PHI_FREE], ph_phi, ctl, a.err)) break;
                        first_phi = false;
                        tc::mbar_arrive_expect_tx(&bar[KB_PHI_FULL], (uint32_t)(SP * RH * 2));
                        for (int kb = 0; kb < RH / 64; ++kb)
                            tc::tma_load_2d(sPHI + kb * SP * 128, &tm_phi, &bar[KB_PHI_FULL], h * RH + kb * 64, phy);
                    }
                }
            }
        } else if (warp == 9) {
            // ---------------- MMA issuer.  X_h = Q W_h^T + P EB_h^T is issued in two parts so that the
            // tensor pipe has work while P is drained and while EB_1 is loaded.  Per chunk:
            //   Q W_0^T -> B;  P EB_0^T -> B;  state_0 += EB_0 K;
            //   Q W_1^T -> A (once P is drained);  P EB_1^T -> A;  s_0 -> B (once Y_0 is out of B);
            //   state_1 += EB_1 K;  s_1 -> B;  P of the next chunk -> A.
            // With one half the scores go to A once P is drained (B holds only RH columns).
            if (lane == 0) {
                uint32_t ph_qk = 0, ph_eb = 0, ph_phi = 0, ph_freeA = 0, ph_freeB = 0, ph_p = 0, ph_w = 0, ph_y = 0;
                const uint32_t id_P = tc::idesc_bf16(128, kC, false, false);
                const uint32_t id_X = tc::idesc_bf16(128, RH, false, false);
                const uint32_t id_S = tc::idesc_bf16(128, S, false, false);
                const uint32_t id_U = tc::idesc_bf16(128, D, false, true);
                const uint32_t accA = tb + colA, accB = tb + colB;
                constexpr bool sB = NH == 2;
                const uint32_t accS = sB ? accB : accA;
                auto peb = [&](uint32_t dX) {
                    // X_h += P EB_h^T
                    mma_steps<false>(dX, sP, kC, sEB, 128, id_X, kC / 16, true);
                    tc::mma_commit(&bar[dX == accA ? KB_ACC_FULL_A : KB_ACC_FULL_B]);
                };
                auto state_update = [&](int h) {
                    // state block h += EB_h (A, 128 rows) . K (B, MN-major)
                    mma_steps<true>(tb + h * D, sEB, 128, sK, kC, id_U, kC / 16, true);
                    tc::mma_commit(&bar[KB_STATE_DONE + h]);
                    tc::mma_commit(&bar[KB_EB_FREE]);
                    if (h == NH - 1) tc::mma_commit(&bar[KB_QK_FREE]);
                };
                auto s_part = [&](int h) -> bool {
                    // s (+)= Y_h PHI_h^T
                    if (!wait_bar(&bar[KB_PHI_FULL], ph_phi, ctl, a.err)) return false;
                    if (!wait_bar(&bar[KB_Y_READY], ph_y, ctl, a.err)) return false;
                    tc::tc_fence_after();
                    mma_steps<false>(accS, sY, kC, sPHI, SP, id_S, RH / 16, h > 0);
                    tc::mma_commit(&bar[KB_Y_FREE]);
                    tc::mma_commit(&bar[KB_PHI_FREE]);
                    return true;
                };
                // P of the first chunk; every later P is issued at the end of the chunk before it
                auto issue_p = [&](bool first) -> bool {
                    if (!wait_bar(&bar[KB_QK_FULL], ph_qk, ctl, a.err)) return false;
                    // A: last read by the previous chunk's Y_1 drain (two halves) or softmax (one half)
                    if (!first && !wait_bar(&bar[KB_ACC_FREE_A], ph_freeA, ctl, a.err)) return false;
                    tc::tc_fence_after();
                    mma_steps<false>(accA, sQ, kC, sK, kC, id_P, D / 16, false);
                    tc::mma_commit(&bar[KB_ACC_FULL_A]);
                    return true;
                };
                bool ok = c_begin < c_end && issue_p(true);
                for (int c = c_begin; c < c_end && ok; ++c) {
                    ok = false;
                    const bool first = c == c_begin;
                    // X_0 -> B: last read by the previous chunk's softmax (two halves) or Y_0 drain (one)
                    if (!wait_bar(&bar[KB_W_READY], ph_w, ctl, a.err)) break;
                    if (!first && !wait_bar(&bar[KB_ACC_FREE_B], ph_freeB, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<false>(accB, sQ, kC, sW, RH, id_X, D / 16, false);
                    tc::mma_commit(&bar[KB_W_FREE]);
                    if (!wait_bar(&bar[KB_EB_FULL], ph_eb, ctl, a.err)) break;
                    if (!wait_bar(&bar[KB_P_READY], ph_p, ctl, a.err)) break;
                    tc::tc_fence_after();
                    peb(accB);
                    state_update(0);
                    if (NH == 2) {
                        // X_1 -> A once P has been drained
                        if (!wait_bar(&bar[KB_W_READY], ph_w, ctl, a.err)) break;
                        if (!wait_bar(&bar[KB_ACC_FREE_A], ph_freeA, ctl, a.err)) break;
                        tc::tc_fence_after();
                        mma_steps<false>(accA, sQ, kC, sW, RH, id_X, D / 16, false);
                        tc::mma_commit(&bar[KB_W_FREE]);
                        if (!wait_bar(&bar[KB_EB_FULL], ph_eb, ctl, a.err)) break;
                        tc::tc_fence_after();
                        peb(accA);
                    }
                    // s_0 once its region has been drained (X_0 into Y, or P)
                    if (sB ? !wait_bar(&bar[KB_ACC_FREE_B], ph_freeB, ctl, a.err)
                           : !wait_bar(&bar[KB_ACC_FREE_A], ph_freeA, ctl, a.err))
                        break;
                    if (!s_part(0)) break;
                    if (NH == 2) {
                        state_update(1);
                        if (!s_part(1)) break;
                    }
                    tc::mma_commit(&bar[sB ? KB_ACC_FULL_B : KB_ACC_FULL_A]);
                    ok = c + 1 >= c_end || issue_p(false);
                }
                tc::mma_commit(&bar[KB_EXIT]);
                uint32_t ph_exit = 0;
                tc::mbar_wait(&bar[KB_EXIT], ph_exit);
            }
        } else if (warp == 10) {
            // ---------------- p store: once the epilogue has written a chunk's probabilities into the
            // Y tile, bulk-store them and hand the tile back when the copy has read it
            if (lane == 0) {
                uint32_t ph_psmem = 0;
                for (int c = c_begin; c < c_end; ++c) {
                    if (!wait_bar(&bar[KB_P_SMEM], ph_psmem, ctl, a.err)) break;
                    for (int kb = 0; kb < SP / 64; ++kb) tc::tma_store_3d(&tm_p, sY + kb * kC * 128, kb * 64, c * kC, bh);
                    tc::bulk_commit();
                    tc::bulk_wait_read0();
                    tc::mbar_arrive(&bar[KB_Y_STORED]);
                }
                tc::bulk_wait0();
            }
        }
    } else {
        tc::reg_alloc<kEpiRegs>();
        {
            // ---------------- epilogue warps 0-7: thread = TMEM lane = token row / state row;
            // warpgroup wg handles columns [wg*N/2, (wg+1)*N/2) of every N-column drain.
            // Per chunk: W_1; Y_0; W_0 of the next chunk; Y_1; softmax; P of the next chunk (one half:
            // Y_0, W_0, softmax, P).
            const int row = threadIdx.x & 127, wg = threadIdx.x >> 7, lane_base = (warp & 3) * 32;
            // softmax partials [2 (max, sum)][2 (warpgroup)][128 rows] in the control area
            float *red = reinterpret_cast<float *>(sm + lay.bars + 1024);
            uint32_t ph_fullA = 0, ph_fullB = 0, ph_wfree = 0, ph_yfree = 0, ph_sync = 0, ph_ystored = 0;
            uint32_t ph_states = 0;   // bit h: phase parity of STATE_DONE + h
            const int M = g.M;
            constexpr int XH = RH / 2;        // X columns per warpgroup (XH/2 modes)
            constexpr int DH = D / 2;         // state columns per warpgroup
            constexpr int SH = S >= 64 ? S / 2 : S;   // slot columns per warpgroup (S = 32: warpgroup 0 only)
            // first mode of this thread's range in each half (two interleaved chains per range), and
            // the drain phases of this row: exact at the CTA's first chunk, then advanced per chunk
            const int m00 = wg * (XH / 2), m10 = RH / 2 + wg * (XH / 2);
            // (the absolute form reads the absolute-frame products as they are: every phase is 1)
            RowPhases rp = row_phases(a.absolute ? 0 : (long long)c_begin * kC + row, m00, m10, NH == 2, hph.w,
                                      hph.tint);
            const RowPhases rp_step = row_phases(a.absolute ? 0 : kC, m00, m10, NH == 2, hph.w, hph.tint);
            // the state is kept in the absolute frame, A = sum_{u < t0} e^{-i m w u} k_u: it needs no
            // rotation between chunks; the carried-in lag-frame state is rotated once
            if (g.NB > 1 && g.G > 1)
                state_prefetch_row<DH>(a.win + ((((size_t)bh * g.G + seg) * 2 + 0) * g.RP + 128) * D + wg * DH, row,
                                       g.R2 - 128, D);
            for (int b = 0; b < g.NB; ++b) {
                const float *src = (g.G > 1) ? a.win + ((((size_t)bh * g.G + seg) * 2 + 0) * g.RP + b * 128) * D : nullptr;
                const float2 f = abs_phase((long long)((b * 128 + row) >> 1) * c_begin * kC, hph.w, hph.tint);
                state_init_abs<DH>(tb, b * D + wg * DH, row, src ? src + wg * DH : nullptr, g.R2 - b * 128, D, f.x, f.y);
            }
            // W_h: state block h after the previous chunk's update (once that update is done), copied from
            // TMEM into the W tile as bf16 once the MMA that read the previous W is done.  Read just before it
            // is stored (nothing waits for it sooner), in 32-column blocks, so that no packed copy is held in
            // registers across the chunk.
            auto w_copy = [&](int h, bool wait_update, bool wait_free) -> bool {
                if (wait_update && !wait_bar(&bar[KB_STATE_DONE + h], ph_states, h, ctl, a.err)) return false;
                if (wait_free && !wait_bar(&bar[KB_W_FREE], ph_wfree, ctl, a.err)) return false;
                tc::tc_fence_after();
#pragma unroll 1
                for (int g0 = 0; g0 < DH; g0 += 32) {
                    float v[32];
                    tc::tmem_ld<32>(tmem_addr(tb, lane_base, h * D + wg * DH + g0), v);
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 32; i += 2) pk[i / 2] = tc::pack_bf16x2(v[i], v[i + 1]);
                    if (row < RH) st_row32_packed(sW, RH, row, wg * DH + g0, pk);
                }
                tc::fence_proxy_async_smem();
                tc::tc_fence_before();
                epi_arrive(&bar[KB_W_READY]);
                return true;
            };
            // Y_h = e^{i m w t} X_h (t = absolute token of this row) from accumulator region `col`,
            // two interleaved mode chains
            auto y_drain = [&](int h, int col, const RowPhases &rp) {
                const float2 pa = h ? rp.h1 : rp.h0, pb = cmul(pa, rp.e1), e2 = rp.e2;
                float ca = pa.x, sa = pa.y, cb = pb.x, sb = pb.y;
                // 32-column blocks in a rolled loop: the epilogue's code per chunk has to stay within the
                // instruction cache, and the phases carry from block to block
#pragma unroll 1
                for (int g0 = 0; g0 < XH; g0 += 32) {
                    float v[32];
                    tc::tmem_ld<32>(tmem_addr(tb, lane_base, col + wg * XH + g0), v);
#pragma unroll
                    for (int i = 0; i < 32; i += 4) {
                        float xr = v[i], xi = v[i + 1];
                        v[i] = ca * xr - sa * xi;
                        v[i + 1] = sa * xr + ca * xi;
                        xr = v[i + 2];
                        xi = v[i + 3];
                        v[i + 2] = cb * xr - sb * xi;
                        v[i + 3] = sb * xr + cb * xi;
                        float t1 = ca * e2.x - sa * e2.y, t2 = sa * e2.x + ca * e2.y;
                        ca = t1;
                        sa = t2;
                        t1 = cb * e2.x - sb * e2.y;
                        t2 = sb * e2.x + cb * e2.y;
                        cb = t1;
                        sb = t2;
                    }
                    st_row32_bf16(sY, kC, row, wg * XH + g0, v);
                }
                tc::fence_proxy_async_smem();
                tc::tc_fence_before();
                epi_arrive(&bar[KB_Y_READY]);
            };
            // P drain: causal mask u <= t, bf16 -> sP
            auto p_drain = [&]() -> bool {
                if (!wait_bar(&bar[KB_ACC_FULL_A], ph_fullA, ctl, a.err)) return false;
                tc::tc_fence_after();
#pragma unroll 1
                for (int g0 = 0; g0 < 64; g0 += 32) {
                    float v[32];
                    tc::tmem_ld<32>(tmem_addr(tb, lane_base, colA + wg * 64 + g0), v);
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (wg * 64 + g0 + i > row) v[i] = 0.f;
                    st_row32_bf16(sP, kC, row, wg * 64 + g0, v);
                }
                tc::fence_proxy_async_smem();
                tc::tc_fence_before();
                epi_arrive(&bar[KB_P_READY]);
                epi_arrive(&bar[KB_ACC_FREE_A]);
                return true;
            };
            // W_0 of the first chunk (the carried-in state as it is) and its P; every W_1 is copied at the
            // start of its chunk
            bool bad = false;
            if (c_begin < c_end) bad = !w_copy(0, false, false) || !p_drain();
            for (int c = c_begin; c < c_end && !bad; ++c) {
                const int t0 = c * kC;
                const int n = min(kC, g.L - t0);
                const bool rot = c > c_begin, more = c + 1 < c_end;
                if (rot) advance(rp, rp_step);
                // W_1 once Q W_0^T has read W_0 (state_1 of the previous chunk's update: this chunk's state_1
                // update waits for W_1, since Q W_1^T reads it)
                if (NH == 2 && !w_copy(1, rot, true)) { bad = true; break; }
                // Y_0 from B; the previous chunk's probabilities must have left the Y tile
                if (!wait_bar(&bar[KB_ACC_FULL_B], ph_fullB, ctl, a.err)) { bad = true; break; }
                if (rot && !wait_bar(&bar[KB_Y_STORED], ph_ystored, ctl, a.err)) { bad = true; break; }
                tc::tc_fence_after();
                y_drain(0, colB, rp);
                epi_arrive(&bar[KB_ACC_FREE_B]);
                // W_0 of the next chunk (the state after this chunk's first update), stored once Q W_1^T (with
                // one half Q W_0^T) has read the W tile: between the two Y drains, where the epilogue would
                // otherwise wait for P EB_1^T and s_0
                if (more && !w_copy(0, true, true)) { bad = true; break; }
                if (NH == 2) {
                    // Y_1 from A once s_0 has read Y_0
                    if (!wait_bar(&bar[KB_ACC_FULL_A], ph_fullA, ctl, a.err)) { bad = true; break; }
                    if (!wait_bar(&bar[KB_Y_FREE], ph_yfree, ctl, a.err)) { bad = true; break; }
                    tc::tc_fence_after();
                    y_drain(1, colA, rp);
                    epi_arrive(&bar[KB_ACC_FREE_A]);
                }
                // masked softmax over the S slots; the two warpgroups exchange their (max, sum) pairs once
                constexpr bool sB = NH == 2;
                if (sB ? !wait_bar(&bar[KB_ACC_FULL_B], ph_fullB, ctl, a.err)
                       : !wait_bar(&bar[KB_ACC_FULL_A], ph_fullA, ctl, a.err)) {
                    bad = true;
                    break;
                }
                if (!wait_bar(&bar[KB_Y_FREE], ph_yfree, ctl, a.err)) { bad = true; break; }
                tc::tc_fence_after();
                {
                    const bool active = wg == 0 || S >= 64;
                    const int j0 = (S >= 64) ? wg * SH : 0;
                    const int t = t0 + row;
                    // slots are visible when t >= D_j; past the largest lag of the grid every slot is
                    const bool all_visible = t0 >= sdelta[S - 1];
                    const float sl2 = a.scale * 1.4426950408889634f;   // scores in log2 units
                    float v[SH];
                    if (active) tc::tmem_ld<SH>(tmem_addr(tb, lane_base, (sB ? colB : colA) + j0), v);
                    tc::tc_fence_before();
                    epi_arrive(&bar[sB ? KB_ACC_FREE_B : KB_ACC_FREE_A]);
                    float mx = -INFINITY, sum = 0.f;
                    if (active) {
                        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                        if (all_visible) {
#pragma unroll
                            for (int j = 0; j < SH; j += 2) {
                                mul2_bcast(v[j], v[j + 1], sl2);
                                m4[j & 3] = fmaxf(m4[j & 3], v[j]);
                                m4[(j + 1) & 3] = fmaxf(m4[(j + 1) & 3], v[j + 1]);
                            }
                        } else {
                            // the lags D_j do not decrease, so the visible slots are j < nvis(t): one
                            // binary search instead of a lag load per slot
                            int lo = 0, hi = S;
                            while (lo < hi) {
                                const int mid = (lo + hi) >> 1;
                                if (sdelta[mid] <= t) lo = mid + 1;
                                else hi = mid;
                            }
                            const int nvis = lo - j0;
#pragma unroll
                            for (int j = 0; j < SH; ++j) {
                                v[j] = (j < nvis) ? v[j] * sl2 : -INFINITY;
                                m4[j & 3] = fmaxf(m4[j & 3], v[j]);
                            }
                        }
                        mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
                        // a half whose slots are all hidden has mx = -inf: exponentiate against 0 instead
                        const float mref = (mx == -INFINITY) ? 0.f : mx;
                        float s4[4] = {0.f, 0.f, 0.f, 0.f};
                        // exponents in pairs through packed fp16 ex2: the probabilities are stored in
                        // bf16, whose resolution (2^-8) is coarser than the fp16 path's error
#pragma unroll
                        for (int j = 0; j < SH; j += 2) {
                            const float2 d2 = sub2_bcast(v[j], v[j + 1], mref);
                            const float2 e2 = tc::exp2_pair_f16(d2.x, d2.y);   // -inf -> 0
                            v[j] = e2.x;
                            v[j + 1] = e2.y;
                            add2(s4[j & 3], s4[(j + 1) & 3], e2.x, e2.y);
                        }
                        sum = (s4[0] + s4[1]) + (s4[2] + s4[3]);
                    }
                    float gmx = mx, gsum = sum;
                    if (S >= 64) {
                        red[wg * 128 + row] = mx;
                        red[256 + wg * 128 + row] = sum;
                        if (!epi_sync(&bar[KB_EPI_SYNC], ph_sync, ctl, a.err)) { bad = true; break; }
                        const float m0 = red[row], m1 = red[128 + row];
                        gmx = fmaxf(m0, m1);
                        gsum = red[256 + row] * exp2f(m0 - gmx) + red[384 + row] * exp2f(m1 - gmx);
                    }
                    if (active) {
                        const float f = exp2f(mx - gmx) / gsum;
#pragma unroll
                        for (int j = 0; j < SH; j += 2) mul2_bcast(v[j], v[j + 1], f);
#pragma unroll
                        for (int g0 = 0; g0 < SH; g0 += 32) st_row32_bf16(sY, kC, row, j0 + g0, v + g0);
                    } else if (SP > S) {
                        float z[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) z[i] = 0.f;
                        for (int g0 = S; g0 < SP; g0 += 32) st_row32_bf16(sY, kC, row, g0, z);
                    }
                    if (wg == 0 && row < n && a.lse) a.lse[(size_t)bh * g.L + t] = (gmx + log2f(gsum)) * 0.6931471805599453f;
                    tc::fence_proxy_async_smem();
                    epi_arrive(&bar[KB_P_SMEM]);
                }
                // the next chunk's P once the softmax has loaded the scores (they free the next chunk's Q W_0^T
                // at once; with one half they also occupy A until then)
                if (more && !p_drain()) { bad = true; break; }

            }
            // final K state (lag frame at t = L-1) after the last chunk of the last segment
            if (!bad && seg == g.G - 1 && a.state_out && c_end > c_begin) {
                for (int h = 0; h < NH; ++h)
                    if (!wait_bar(&bar[KB_STATE_DONE + h], ph_states, h, ctl, a.err)) { bad = true; break; }
                if (!bad) {
                    tc::tc_fence_after();
                    for (int b = 0; b < g.NB; ++b) {
                        const int r = b * 128 + row, m = r >> 1;
                        float *dst = (r < g.R2) ? a.state_out + ((size_t)bh * 2 * g.R2 + r) * D : nullptr;
                        const float2 f =
                            (m < M) ? abs_phase((long long)m * (g.L - 1), hph.w, hph.tint) : make_float2(1.f, 0.f);
                        state_pass<DH>(tb, b * D + wg * DH, row, true, f.x, f.y, false, nullptr, 0, dst, wg * DH);
                    }
                }
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, ncols);
    }
}

// ================================================================== V pass

struct VLayout {
    size_t v, y0, a1, bx, bz, w, phi, bars, total;
};

// Every 128-row tile buffer holds 32 KB: p (128 x SP), G (128 x C), EB_h (128 x C), A'_h
// (128 x RH), W_h (RH x d) or O (128 x d).
__host__ __device__ inline VLayout v_layout(const Geo &g) {
    VLayout l;
    size_t off = 0;
    const size_t tile = (size_t)kC * 128 * 2;
    l.v = off;   off += (size_t)kC * g.D * 2;
    l.y0 = off;  off += tile;   // A'_0, then the staged output tile
    l.a1 = off;  off += tile;   // A'_1
    l.bx = off;  off += tile;   // p then G, and EB_0, alternating with bz from chunk to chunk
    l.bz = off;  off += tile;
    l.w = off;   off += tile;   // W_0
    l.phi = off; off += tile;   // PHI_0, PHI_1, EB_1, then W_1
    l.bars = off; off += 1024;
    l.total = off + 1024;
    return l;
}

// One barrier per hand-off (see the K pass).  A'_0 / A'_1 and W_0 / W_1 each have their own ready
// barrier: the second of each pair can be signalled before the MMA issuer has waited for the first.
enum VBar {
    VB_P_FULL, VB_P_FREE, VB_V_FULL, VB_V_FREE, VB_EB_FULL, VB_EB_FREE, VB_PH_FULL, VB_PH_FREE,
    VB_U_FULL, VB_U_FREE, VB_G_FULL, VB_G_FREE, VB_A_READY, VB_A_READY1, VB_G_READY, VB_W_READY, VB_W_READY1, VB_W_FREE,
    VB_STATE_DONE, VB_STATE_DONE1, VB_STATE_READ, VB_O_FULL, VB_O_SMEM, VB_O_STORED, VB_EXIT, VB_COUNT
};

// V pass.  Per chunk and mode half h: U_h = p PHI_h; A'_h = e^{-i m w t} U_h (t absolute) into shared
// memory; G = sum_h A'_h EB_h (causal mask on drain, written over p); state_h += EB_h V; and
// O = sum_h A'_h W_h + G V.  Buffers: A'_0 and the staged output in y0, A'_1 in a1; p/G and EB_0
// alternate between bx and bz from chunk to chunk, so the next chunk's p loads into this chunk's
// EB_0 buffer as soon as state_0 has read it; the PHI tile takes EB_1 once U_1 has read PHI_1, and
// W_1 once state_1 has read EB_1, so O = A'_0 W_0 + A'_1 W_1 runs without a wait in between.
template <int D, int RH, int NH>
__global__ void __launch_bounds__(kPassThreads, 1)
    k_vpass(const __grid_constant__ CUtensorMap tm_p, const __grid_constant__ CUtensorMap tm_v,
            const __grid_constant__ CUtensorMap tm_eb, const __grid_constant__ CUtensorMap tm_phi,
            const __grid_constant__ CUtensorMap tm_o, Args a) {
    const Geo &g = a.g;
    // heads fastest: the CTAs of one segment run in the same wave and share its EB tables in L2
    const int bh = blockIdx.x % g.BH, seg = blockIdx.x / g.BH;
    const int c_begin = seg * g.cps, c_end = min(g.nchunks, c_begin + g.cps);
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const VLayout lay = v_layout(g);
    uint8_t *sV = sm + lay.v, *sY0 = sm + lay.y0, *sA1 = sm + lay.a1, *sBX = sm + lay.bx, *sBZ = sm + lay.bz;
    uint8_t *sW = sm + lay.w, *sPHI = sm + lay.phi;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + lay.bars);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + VB_COUNT);
    Ctl *ctl = reinterpret_cast<Ctl *>(bar + VB_COUNT + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int SP = g.SP;
    // chunk i (from c_begin) keeps p/G in pbuf(i) and EB_0 in ebuf(i), alternating
    auto pbuf = [&](int i) { return (i & 1) ? sBZ : sBX; };
    auto ebuf = [&](int i) { return (i & 1) ? sBX : sBZ; };
    // TMEM: [0, NB*D) state; colU (128 cols: U_h, then O); colG (128 cols).
    const int colU = g.NB * D, colG = colU + 128;
    const uint32_t ncols = (uint32_t)(colG + 128) <= 256 ? 256u : 512u;  // host: pow2_cols(NB*D + 256)

    if (threadIdx.x == 0) {
        for (int i = 0; i < VB_COUNT; ++i) {
            const bool epi = i == VB_U_FREE || i == VB_G_FREE || i == VB_A_READY || i == VB_A_READY1 || i == VB_G_READY ||
                             i == VB_W_READY || i == VB_W_READY1 || i == VB_STATE_READ || i == VB_O_SMEM;
            tc::mbar_init(&bar[i], epi ? kPassEpiWarps : 1);
        }
        ctl->abort = 0;
        ctl->kernel = 3;
        ctl->bar0 = bar;
        tc::fence_barrier_init();
    }
    if (warp == 9) { tc::tmem_alloc(tslot, ncols); tc::tmem_relinquish(); }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tb = *tslot;
    tc::pdl_wait();      // p from the K pass, and the tables and states before it
    const HeadW hph = head_w(a, bh);                      // this head's w and integer period
    const int eby = (bh % a.H) * a.eb_rows_h, phy = (bh % a.H) * a.phi_rows_h;   // its table rows

    if (warp >= 8) {
        if (warp == 8) {
            // ---------------- TMA producer, in the order of first use: p, PHI_0, EB_0, V, PHI_1, EB_1
            if (lane == 0) {
                tc::tma_prefetch_desc(&tm_p); tc::tma_prefetch_desc(&tm_v);
                tc::tma_prefetch_desc(&tm_eb); tc::tma_prefetch_desc(&tm_phi);
                uint32_t ph_p = 0, ph_v = 0, ph_eb = 0, ph_ph = 0;
                for (int c = c_begin; c < c_end; ++c) {
                    const int i = c - c_begin;
                    const bool first = i == 0;
                    // p: the buffer held the previous chunk's EB_0 (freed once state_0 has read it)
                    if (!first && !wait_bar(&bar[VB_P_FREE], ph_p, ctl, a.err)) break;
                    tc::mbar_arrive_expect_tx(&bar[VB_P_FULL], (uint32_t)(kC * SP * 2));
                    for (int kb = 0; kb < SP / 64; ++kb)
                        tc::tma_load_3d(pbuf(i) + kb * kC * 128, &tm_p, &bar[VB_P_FULL], kb * 64, c * kC, bh);
                    // PHI_0 (the PHI tile last held the previous chunk's W_1, or PHI_0 with one half)
                    if (!first && !wait_bar(&bar[VB_PH_FREE], ph_ph, ctl, a.err)) break;
                    tc::mbar_arrive_expect_tx(&bar[VB_PH_FULL], (uint32_t)(SP * RH * 2));
                    for (int kb = 0; kb < RH / 64; ++kb)
                        tc::tma_load_2d(sPHI + kb * SP * 128, &tm_phi, &bar[VB_PH_FULL], kb * 64, phy);
                    // EB_0 into the buffer of the previous chunk's p/G (freed once G V has read it)
                    if (!first && !wait_bar(&bar[VB_EB_FREE], ph_eb, ctl, a.err)) break;
                    tc::mbar_arrive_expect_tx(&bar[VB_EB_FULL], (uint32_t)(128 * kC * 2));
                    for (int kb = 0; kb < 2; ++kb)
                        tc::tma_load_2d(ebuf(i) + kb * 128 * 128, &tm_eb, &bar[VB_EB_FULL], kb * 64, eby + c * g.RP);
                    if (!first && !wait_bar(&bar[VB_V_FREE], ph_v, ctl, a.err)) break;
                    tc::mbar_arrive_expect_tx(&bar[VB_V_FULL], (uint32_t)(kC * D * 2));
                    for (int db = 0; db < D / 64; ++db)
                        tc::tma_load_3d(sV + db * kC * 128, &tm_v, &bar[VB_V_FULL], db * 64, c * kC, bh);
                    if (NH == 2) {
                        // PHI_1 once U_0 has read PHI_0; EB_1 into the PHI tile once U_1 has read PHI_1
                        if (!wait_bar(&bar[VB_PH_FREE], ph_ph, ctl, a.err)) break;
                        tc::mbar_arrive_expect_tx(&bar[VB_PH_FULL], (uint32_t)(SP * RH * 2));
                        for (int kb = 0; kb < RH / 64; ++kb)
                            tc::tma_load_2d(sPHI + kb * SP * 128, &tm_phi, &bar[VB_PH_FULL], RH + kb * 64, phy);
                        if (!wait_bar(&bar[VB_PH_FREE], ph_ph, ctl, a.err)) break;
                        tc::mbar_arrive_expect_tx(&bar[VB_PH_FULL], (uint32_t)(128 * kC * 2));
                        for (int kb = 0; kb < 2; ++kb)
                            tc::tma_load_2d(sPHI + kb * 128 * 128, &tm_eb, &bar[VB_PH_FULL], kb * 64,
                                            eby + c * g.RP + 128);
                    }
                }
            }
        } else if (warp == 9) {
            // ---------------- MMA issuer.  Per chunk: U_0; state_0 += EB_0 V; U_1 (once A'_0 is drained);
            // G = A'_0 EB_0; G += A'_1 EB_1; state_1 += EB_1 V; O = A'_0 W_0 (+ A'_1 W_1); O += G V.
            if (lane == 0) {
                uint32_t ph_p = 0, ph_v = 0, ph_eb = 0, ph_ph = 0, ph_ufree = 0, ph_gfree = 0, ph_a0 = 0, ph_a1 = 0, ph_gready = 0;
                uint32_t ph_w0 = 0, ph_w1 = 0, ph_sread = 0;
                const uint32_t id_U = tc::idesc_bf16(128, RH, false, true);
                const uint32_t id_G = tc::idesc_bf16(128, kC, false, true);
                const uint32_t id_O = tc::idesc_bf16(128, D, false, true);
                const uint32_t accU = tb + colU, accG = tb + colG;
                for (int c = c_begin; c < c_end; ++c) {
                    const int i = c - c_begin;
                    const bool first = i == 0;
                    uint8_t *sP = pbuf(i), *sE0 = ebuf(i);
                    // U_0 -> U (last read by the previous chunk's O drain)
                    if (!wait_bar(&bar[VB_P_FULL], ph_p, ctl, a.err)) break;
                    if (!wait_bar(&bar[VB_PH_FULL], ph_ph, ctl, a.err)) break;
                    if (!first && !wait_bar(&bar[VB_U_FREE], ph_ufree, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<true>(accU, sP, kC, sPHI, SP, id_U, SP / 16, false);
                    tc::mma_commit(&bar[VB_U_FULL]);
                    tc::mma_commit(&bar[VB_PH_FREE]);
                    // state_0 += EB_0 V once this chunk's W tiles have been read from the state: it needs
                    // neither A' nor G, so it runs while A'_0 is drained
                    if (!wait_bar(&bar[VB_EB_FULL], ph_eb, ctl, a.err)) break;
                    if (!wait_bar(&bar[VB_STATE_READ], ph_sread, ctl, a.err)) break;
                    if (!wait_bar(&bar[VB_V_FULL], ph_v, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<true>(tb, sE0, 128, sV, kC, id_O, kC / 16, true);
                    tc::mma_commit(&bar[VB_STATE_DONE]);
                    if (NH == 2) {
                        // U_1 -> U once A'_0 is drained
                        if (!wait_bar(&bar[VB_PH_FULL], ph_ph, ctl, a.err)) break;
                        if (!wait_bar(&bar[VB_U_FREE], ph_ufree, ctl, a.err)) break;
                        tc::tc_fence_after();
                        mma_steps<true>(accU, sP, kC, sPHI, SP, id_U, SP / 16, false);
                        tc::mma_commit(&bar[VB_U_FULL]);
                        tc::mma_commit(&bar[VB_PH_FREE]);
                    }
                    // G = A'_0 EB_0 -> G (last read by the previous chunk's G drain)
                    if (!wait_bar(&bar[VB_A_READY], ph_a0, ctl, a.err)) break;
                    if (!first && !wait_bar(&bar[VB_G_FREE], ph_gfree, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<true>(accG, sY0, kC, sE0, 128, id_G, RH / 16, false);
                    if (NH == 1) tc::mma_commit(&bar[VB_G_FULL]);
                    tc::mma_commit(&bar[VB_P_FREE]);   // EB_0's buffer takes the next chunk's p
                    if (NH == 2) {
                        // G += A'_1 EB_1 (EB_1 in the PHI tile); state_1 += EB_1 V
                        if (!wait_bar(&bar[VB_A_READY1], ph_a1, ctl, a.err)) break;
                        if (!wait_bar(&bar[VB_PH_FULL], ph_ph, ctl, a.err)) break;
                        tc::tc_fence_after();
                        mma_steps<true>(accG, sA1, kC, sPHI, 128, id_G, RH / 16, true);
                        tc::mma_commit(&bar[VB_G_FULL]);
                        mma_steps<true>(tb + D, sPHI, 128, sV, kC, id_O, kC / 16, true);
                        tc::mma_commit(&bar[VB_STATE_DONE1]);   // the PHI tile may take W_1
                    }
                    // O = A'_0 W_0 -> U once the last A' has been drained
                    if (!wait_bar(&bar[VB_U_FREE], ph_ufree, ctl, a.err)) break;
                    if (!wait_bar(&bar[VB_W_READY], ph_w0, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<true>(accU, sY0, kC, sW, RH, id_O, RH / 16, false);
                    tc::mma_commit(&bar[VB_W_FREE]);
                    if (NH == 2) {
                        // O += A'_1 W_1 (W_1 in the PHI tile, which then takes the next PHI_0)
                        if (!wait_bar(&bar[VB_W_READY1], ph_w1, ctl, a.err)) break;
                        tc::tc_fence_after();
                        mma_steps<true>(accU, sA1, kC, sPHI, RH, id_O, RH / 16, true);
                        tc::mma_commit(&bar[VB_PH_FREE]);
                    }
                    // O += G V (G written over p by the epilogue)
                    if (!wait_bar(&bar[VB_G_READY], ph_gready, ctl, a.err)) break;
                    tc::tc_fence_after();
                    mma_steps<true>(accU, sP, kC, sV, kC, id_O, kC / 16, true);
                    tc::mma_commit(&bar[VB_O_FULL]);
                    tc::mma_commit(&bar[VB_V_FREE]);
                    tc::mma_commit(&bar[VB_EB_FREE]);   // p/G's buffer takes the next chunk's EB_0
                }
                tc::mma_commit(&bar[VB_EXIT]);
                uint32_t ph_exit = 0;
                tc::mbar_wait(&bar[VB_EXIT], ph_exit);
            }
        } else if (warp == 10) {
            // ---------------- O store: bulk-store each output tile staged in y0 and hand the buffer
            // back once the copy has read it
            if (lane == 0) {
                uint32_t ph_osmem = 0;
                for (int c = c_begin; c < c_end; ++c) {
                    if (!wait_bar(&bar[VB_O_SMEM], ph_osmem, ctl, a.err)) break;
                    for (int db = 0; db < D / 64; ++db) tc::tma_store_3d(&tm_o, sY0 + db * kC * 128, db * 64, c * kC, bh);
                    tc::bulk_commit();
                    tc::bulk_wait_read0();
                    tc::mbar_arrive(&bar[VB_O_STORED]);
                }
                tc::bulk_wait0();
            }
        }
    } else {
        {
            // ---------------- epilogue warps 0-7 (thread = TMEM lane = token row / state row; warpgroup
            // wg handles half of the columns of every drain).  Per chunk: read W_0, W_1 from the state
            // (letting the state updates proceed) and store W_0; A'_0; A'_1; W_1; G; O.
            const int row = threadIdx.x & 127, wg = threadIdx.x >> 7, lane_base = (warp & 3) * 32;
            const int M = g.M;
            constexpr int XH = RH / 2, DH = D / 2;
            uint32_t ph_u = 0, ph_g = 0, ph_wfree = 0, ph_o = 0, ph_ostored = 0;
            uint32_t ph_states = 0;   // bit h: phase parity of STATE_DONE + h
            // first mode of this thread's range in each half, and the drain phases of this row
            const int m00 = wg * (XH / 2), m10 = RH / 2 + wg * (XH / 2);
            RowPhases rp = row_phases(a.absolute ? 0 : (long long)c_begin * kC + row, m00, m10, NH == 2, hph.w,
                                      hph.tint);
            const RowPhases rp_step = row_phases(a.absolute ? 0 : kC, m00, m10, NH == 2, hph.w, hph.tint);
            // V state in the absolute frame (see the K pass)
            if (g.NB > 1 && g.G > 1)
                state_prefetch_row<DH>(a.win + ((((size_t)bh * g.G + seg) * 2 + 1) * g.RP + 128) * D + wg * DH, row,
                                       g.R2 - 128, D);
            for (int b = 0; b < g.NB; ++b) {
                const float *src = (g.G > 1) ? a.win + ((((size_t)bh * g.G + seg) * 2 + 1) * g.RP + b * 128) * D : nullptr;
                const float2 f = abs_phase((long long)((b * 128 + row) >> 1) * c_begin * kC, hph.w, hph.tint);
                state_init_abs<DH>(tb, b * D + wg * DH, row, src ? src + wg * DH : nullptr, g.R2 - b * 128, D, f.x, f.y);
            }
            // W_0 goes to the W tile once the previous chunk's O = A'_0 W_0 has read it; W_1 goes to the
            // PHI tile once state_1 has read EB_1 there
            auto w_store = [&](int h, bool wait_free, const uint32_t *pk) -> bool {
                if (h == 0 && wait_free && !wait_bar(&bar[VB_W_FREE], ph_wfree, ctl, a.err)) return false;
                if (h == 1 && !wait_bar(&bar[VB_STATE_DONE1], ph_states, 1, ctl, a.err)) return false;
                uint8_t *dst = h ? sPHI : sW;
                if (row < RH) {
#pragma unroll
                    for (int g0 = 0; g0 < DH; g0 += 32) st_row32_packed(dst, RH, row, wg * DH + g0, pk + g0 / 2);
                }
                tc::fence_proxy_async_smem();
                tc::tc_fence_before();
                epi_arrive(&bar[VB_W_READY + h]);
                return true;
            };
            bool bad = false;
            for (int c = c_begin; c < c_end && !bad; ++c) {
                const int i = c - c_begin;
                const bool rot = i > 0;
                if (rot) advance(rp, rp_step);
                // W_h: the V state before this chunk's update, into registers (state_1's previous update
                // was awaited before the previous chunk's W_1 store)
                uint32_t pk0[DH / 2], pk1[DH / 2];
                if (rot && !wait_bar(&bar[VB_STATE_DONE], ph_states, 0, ctl, a.err)) break;
                tc::tc_fence_after();
                state_pack<DH>(tb, wg * DH, row, pk0);
                if (NH == 2) state_pack<DH>(tb, D + wg * DH, row, pk1);
                tc::tc_fence_before();
                epi_arrive(&bar[VB_STATE_READ]);
                if (!w_store(0, rot, pk0)) { bad = true; break; }
                // A'_h = e^{-i m w t} U_h (t absolute); y0 held the previous chunk's output tile until
                // the store read it
                if (rot && !wait_bar(&bar[VB_O_STORED], ph_ostored, ctl, a.err)) break;
#pragma unroll
                for (int h = 0; h < NH; ++h) {
                    if (!wait_bar(&bar[VB_U_FULL], ph_u, ctl, a.err)) { bad = true; break; }
                    tc::tc_fence_after();
                    float v[XH];
                    tc::tmem_ld<XH>(tmem_addr(tb, lane_base, colU + wg * XH), v);
                    tc::tc_fence_before();
                    epi_arrive(&bar[VB_U_FREE]);
                    const float2 pa = h ? rp.h1 : rp.h0, pb = cmul(pa, rp.e1), e2 = rp.e2;
                    float ca = pa.x, sa = pa.y, cb = pb.x, sb = pb.y;
#pragma unroll
                    for (int q = 0; q < XH; q += 4) {
                        float uc = v[q], us = v[q + 1];
                        v[q] = ca * uc + sa * us;
                        v[q + 1] = ca * us - sa * uc;
                        uc = v[q + 2];
                        us = v[q + 3];
                        v[q + 2] = cb * uc + sb * us;
                        v[q + 3] = cb * us - sb * uc;
                        float t1 = ca * e2.x - sa * e2.y, t2 = sa * e2.x + ca * e2.y;
                        ca = t1;
                        sa = t2;
                        t1 = cb * e2.x - sb * e2.y;
                        t2 = sb * e2.x + cb * e2.y;
                        cb = t1;
                        sb = t2;
                    }
                    uint8_t *dstA = h ? sA1 : sY0;
#pragma unroll
                    for (int g0 = 0; g0 < XH; g0 += 32) st_row32_bf16(dstA, kC, row, wg * XH + g0, v + g0);
                    tc::fence_proxy_async_smem();
                    epi_arrive(&bar[VB_A_READY + h]);
                }
                if (bad) break;
                // W_1 into the PHI tile once state_1 has read EB_1 there
                if (NH == 2 && !w_store(1, true, pk1)) { bad = true; break; }
                // G drain -> causal mask -> bf16 over p (U_0 and U_1 are done once G is full)
                if (!wait_bar(&bar[VB_G_FULL], ph_g, ctl, a.err)) break;
                tc::tc_fence_after();
                {
                    float v[64];
                    tc::tmem_ld<64>(tmem_addr(tb, lane_base, colG + wg * 64), v);
#pragma unroll
                    for (int q = 0; q < 64; ++q)
                        if (wg * 64 + q > row) v[q] = 0.f;
#pragma unroll
                    for (int g0 = 0; g0 < 64; g0 += 32) st_row32_bf16(pbuf(i), kC, row, wg * 64 + g0, v + g0);
                }
                tc::fence_proxy_async_smem();
                tc::tc_fence_before();
                epi_arrive(&bar[VB_G_READY]);
                epi_arrive(&bar[VB_G_FREE]);
                // O drain -> staged in y0 for the store warp
                if (!wait_bar(&bar[VB_O_FULL], ph_o, ctl, a.err)) break;
                tc::tc_fence_after();
                {
                    float v[DH];
                    tc::tmem_ld<DH>(tmem_addr(tb, lane_base, colU + wg * DH), v);
                    tc::tc_fence_before();
                    epi_arrive(&bar[VB_U_FREE]);
#pragma unroll
                    for (int g0 = 0; g0 < DH; g0 += 32) st_row32_bf16(sY0, kC, row, wg * DH + g0, v + g0);
                    tc::fence_proxy_async_smem();
                    epi_arrive(&bar[VB_O_SMEM]);
                }
            }
            if (!bad && seg == g.G - 1 && a.state_out && c_end > c_begin) {
                // the last chunk's state_1 update was awaited before its W_1 store
                if (!wait_bar(&bar[VB_STATE_DONE], ph_states, 0, ctl, a.err)) bad = true;
                if (!bad) {
                    tc::tc_fence_after();
                    for (int b = 0; b < g.NB; ++b) {
                        const int r = b * 128 + row, m = r >> 1;
                        float *dst = (r < g.R2) ? a.state_out + ((size_t)bh * 2 * g.R2 + g.R2 + r) * D : nullptr;
                        const float2 f =
                            (m < M) ? abs_phase((long long)m * (g.L - 1), hph.w, hph.tint) : make_float2(1.f, 0.f);
                        state_pass<DH>(tb, b * D + wg * DH, row, true, f.x, f.y, false, nullptr, 0, dst, wg * DH);
                    }
                }
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tb, ncols);
    }
}

}  // namespace

// ================================================================== host side

// The period as an integer when w = 2 pi / T and T is a whole number below 2^24 (exact phase
// reduction applies), else 0.
static int integer_period(double T, double w) {
    const double kPi2 = 6.283185307179586;
    if (T >= 16777216.0 || T != floor(T)) return 0;
    if (fabs(w - kPi2 / T) > 1e-15 * kPi2 / T) return 0;
    return (int)T;
}
static int integer_period(const OpDims &d) { return integer_period(d.T, d.w); }

cudaError_t build_bf16_tables(const OpDims &d, int RP, int SP, bf16 *eb, bf16 *phi, cudaStream_t st) {
    long long total = (long long)(RP / 2) * (kC / 8) + (long long)SP * d.R2 + 1;
    int blocks = (int)((total + 255) / 256);
    if (blocks > 2048) blocks = 2048;
    HeadPeriods hp;
    hp.n = 0;
    HeadTint ht = {};
    ProfScope ps(BLA_K_TABLES_BF16, st);
    k_tables_bf16<<<blocks, 256, 0, st>>>(d.M, d.S, SP, RP, 1, 1, hp, ht, d.T, d.w, integer_period(d),
                                          d.absolute ? -1.f : 1.f, eb, phi, nullptr, nullptr, nullptr, nullptr, 0);
    return cudaGetLastError();
}

const char *fwd_bf16_unsupported(const OpDims &d) {
    if (d.dk != d.dv) return "d_k must equal d_v";
    if (d.dk != 64 && d.dk != 128) return "d_k must be 64 or 128";
    if (d.R2 != 64 && d.R2 != 128 && d.R2 != 256) return "2M must be 64, 128 or 256";
    if (d.S != 32 && d.S != 64 && d.S != 128) return "S must be 32, 64 or 128";
    if (d.S > (d.R2 < 64 ? 64 : d.R2)) return "S must not exceed max(2M, 64)";
    if (d.L > (1 << 26)) return "L must not exceed 2^26 tokens (table indices are 32-bit)";
    return nullptr;
}

size_t fwd_bf16_workspace_bytes(const OpDims &d) {
    if (fwd_bf16_unsupported(d)) return 0;
    Geo g = make_geo(d);
    return ws_layout(d, g).total;
}

// Dynamic shared memory to request: at least `bytes`, and when the kernel allocates all 512
// TMEM columns, enough to keep a second CTA of it off the same SM.
static int smem_request(size_t bytes, int tmem_cols) {
    const size_t one_per_sm = 120 * 1024;
    if (tmem_cols >= 512 && bytes < one_per_sm) bytes = one_per_sm;
    return (int)bytes;
}

static int pow2_cols(int n) { return n <= 32 ? 32 : n <= 64 ? 64 : n <= 128 ? 128 : n <= 256 ? 256 : 512; }

// The pass kernels move registers between warpgroups (setmaxnreg); an increase that the launch
// cannot cover would wait forever, so launch only if every thread starts with kLaunchRegs.
static cudaError_t check_register_split(const void *fn) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, fn);
    if (e != cudaSuccess) return e;
    if (fa.numRegs < kLaunchRegs || fa.maxThreadsPerBlock < kPassThreads) return cudaErrorLaunchOutOfResources;
    return cudaSuccess;
}


template <int D, int RH, int S, int NH>
static cudaError_t launch_kpass_n(int smem, int nblk, cudaStream_t st, const CUtensorMap &tq, const CUtensorMap &tk,
                                  const CUtensorMap &teb, const CUtensorMap &tphi, const CUtensorMap &tp, const Args &a) {
    cudaError_t e = cudaFuncSetAttribute(k_kpass<D, RH, S, NH>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    if ((e = check_register_split((const void *)k_kpass<D, RH, S, NH>)) != cudaSuccess) return e;
    ProfScope ps(BLA_K_KPASS, st);
    e = launch_pdl(k_kpass<D, RH, S, NH>, dim3(nblk), dim3(kPassThreads), smem, st, tq, tk, teb, tphi, tp, a);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <int D, int RH, int S>
static cudaError_t launch_kpass_t(int smem, int nblk, cudaStream_t st, const CUtensorMap &tq, const CUtensorMap &tk,
                                  const CUtensorMap &teb, const CUtensorMap &tphi, const CUtensorMap &tp, const Args &a) {
    if constexpr (RH == 128) {
        if (a.g.NH == 2) return launch_kpass_n<D, RH, S, 2>(smem, nblk, st, tq, tk, teb, tphi, tp, a);
    }
    return launch_kpass_n<D, RH, S, 1>(smem, nblk, st, tq, tk, teb, tphi, tp, a);
}

template <int D, int RH>
static cudaError_t launch_kpass_s(const Geo &g, int smem, int nblk, cudaStream_t st, const CUtensorMap &tq,
                                  const CUtensorMap &tk, const CUtensorMap &teb, const CUtensorMap &tphi,
                                  const CUtensorMap &tp, const Args &a) {
    switch (g.S) {
    case 32: return launch_kpass_t<D, RH, 32>(smem, nblk, st, tq, tk, teb, tphi, tp, a);
    case 64: return launch_kpass_t<D, RH, 64>(smem, nblk, st, tq, tk, teb, tphi, tp, a);
    case 128: return launch_kpass_t<D, RH, 128>(smem, nblk, st, tq, tk, teb, tphi, tp, a);
    default: return cudaErrorInvalidValue;
    }
}

static cudaError_t launch_kpass(const Geo &g, int smem, int nblk, cudaStream_t st, const CUtensorMap &tq,
                                const CUtensorMap &tk, const CUtensorMap &teb, const CUtensorMap &tphi,
                                const CUtensorMap &tp, const Args &a) {
    if (g.D == 64 && g.RH == 64) return launch_kpass_s<64, 64>(g, smem, nblk, st, tq, tk, teb, tphi, tp, a);
    if (g.D == 64 && g.RH == 128) return launch_kpass_s<64, 128>(g, smem, nblk, st, tq, tk, teb, tphi, tp, a);
    if (g.D == 128 && g.RH == 64) return launch_kpass_s<128, 64>(g, smem, nblk, st, tq, tk, teb, tphi, tp, a);
    if (g.D == 128 && g.RH == 128) return launch_kpass_s<128, 128>(g, smem, nblk, st, tq, tk, teb, tphi, tp, a);
    return cudaErrorInvalidValue;
}

template <int D, int RH, int NH>
static cudaError_t launch_vpass_n(int smem, int nblk, cudaStream_t st, const CUtensorMap &tp, const CUtensorMap &tv,
                                  const CUtensorMap &teb, const CUtensorMap &tphi, const CUtensorMap &to,
                                  const Args &a) {
    cudaError_t e = cudaFuncSetAttribute(k_vpass<D, RH, NH>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    ProfScope ps(BLA_K_VPASS, st);
    e = launch_pdl(k_vpass<D, RH, NH>, dim3(nblk), dim3(kPassThreads), smem, st, tp, tv, teb, tphi, to, a);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <int D, int RH>
static cudaError_t launch_vpass_t(int smem, int nblk, cudaStream_t st, const CUtensorMap &tp, const CUtensorMap &tv,
                                  const CUtensorMap &teb, const CUtensorMap &tphi, const CUtensorMap &to,
                                  const Args &a) {
    if constexpr (RH == 128) {
        if (a.g.NH == 2) return launch_vpass_n<D, RH, 2>(smem, nblk, st, tp, tv, teb, tphi, to, a);
    }
    return launch_vpass_n<D, RH, 1>(smem, nblk, st, tp, tv, teb, tphi, to, a);
}

static cudaError_t launch_vpass(const Geo &g, int smem, int nblk, cudaStream_t st, const CUtensorMap &tp,
                                const CUtensorMap &tv, const CUtensorMap &teb, const CUtensorMap &tphi,
                                const CUtensorMap &to, const Args &a) {
    if (g.D == 64 && g.RH == 64) return launch_vpass_t<64, 64>(smem, nblk, st, tp, tv, teb, tphi, to, a);
    if (g.D == 64 && g.RH == 128) return launch_vpass_t<64, 128>(smem, nblk, st, tp, tv, teb, tphi, to, a);
    if (g.D == 128 && g.RH == 64) return launch_vpass_t<128, 64>(smem, nblk, st, tp, tv, teb, tphi, to, a);
    if (g.D == 128 && g.RH == 128) return launch_vpass_t<128, 128>(smem, nblk, st, tp, tv, teb, tphi, to, a);
    return cudaErrorInvalidValue;
}

cudaError_t fwd_bf16_run(const OpDims &d, const void *q, const void *k, const void *v, void *o, float *lse,
                         float *state_out, void *workspace, cudaStream_t st) {
    Geo g = make_geo(d);
    if (g.L == 0) {
        if (state_out)
            return cudaMemsetAsync(state_out, 0, sizeof(float) * (size_t)g.BH * 2 * g.R2 * g.D, st);
        return cudaSuccess;
    }
    WsLayout wl = ws_layout(d, g);
    char *ws = static_cast<char *>(workspace);
    cudaError_t e;
    bf16 *eb = reinterpret_cast<bf16 *>(ws + wl.eb), *phi = reinterpret_cast<bf16 *>(ws + wl.phi);
    bf16 *fseg = g.G > 1 ? reinterpret_cast<bf16 *>(ws + wl.fseg) : nullptr;
    int *delta = reinterpret_cast<int *>(ws + wl.delta);
    double *hw = d.periods ? reinterpret_cast<double *>(ws + wl.hw) : nullptr;
    int *htint = d.periods ? reinterpret_cast<int *>(ws + wl.htint) : nullptr;
    // per-head periods: every head's (T_h, w_h) and integer period; nh tables
    HeadPeriods hp;
    head_periods(d, d.omega_in, &hp);
    HeadTint ht;
    for (int h = 0; h < hp.n; ++h) ht.t[h] = integer_period(hp.T[h], hp.w[h]);
    const int nh = hp.n > 0 ? hp.n : 1;
    {
        // EB of every chunk (absolute phases), PHI, FSEG and the slot lags in one launch; with segments
        // the prepass writes EB instead
        const int eb_skip = g.G > 1 ? 1 : 0;
        const long long total = nh * ((eb_skip ? 0 : (long long)g.nchunks * (g.RP / 2) * (kC / 8)) +
                                      (long long)g.SP * g.R2 +
                                      (fseg ? (long long)(g.RP / 2) * ((g.Lseg + 7) / 8) : 0) + g.S + 1);
        const int blocks = (int)(total < 4096 * 256 ? (total + 255) / 256 : 4096);
        ProfScope ps(BLA_K_TABLES_BF16, st);
        k_tables_bf16<<<blocks, 256, 0, st>>>(g.M, g.S, g.SP, g.RP, g.Lseg, g.nchunks, hp, ht, d.T, d.w,
                                              integer_period(d), d.absolute ? -1.f : 1.f, eb, phi, fseg, delta, hw,
                                              htint, eb_skip);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    Args a;
    a.g = g;
    a.scale = d.scale;
    a.w = d.w;
    a.delta = delta;
    a.deltas = g.G > 1 ? reinterpret_cast<float *>(ws + wl.deltas) : nullptr;
    a.deltas_out = const_cast<float *>(a.deltas);
    a.win = g.G > 1 ? reinterpret_cast<float *>(ws + wl.win) : nullptr;
    a.pbuf = reinterpret_cast<bf16 *>(ws + wl.pbuf);
    a.lse = lse;
    a.o = static_cast<bf16 *>(o);
    a.state_out = state_out;
    a.tint = integer_period(d);
    a.absolute = d.absolute;
    a.err = device_error_word();
    a.H = d.H;
    a.eb_rows_h = hp.n > 0 ? g.nchunks * g.RP : 0;
    a.phi_rows_h = hp.n > 0 ? g.SP : 0;
    a.f_rows_h = hp.n > 0 ? g.RP : 0;
    a.delta_h = hp.n > 0 ? g.S : 0;
    a.hw = hw;
    a.htint = htint;
    a.eb_gen = g.G > 1 ? eb : nullptr;
    a.eb_nh = nh;

    // tensor maps
    CUtensorMap tq, tk, tv, tp, teb, tphi, tf, tdl;
    const uint64_t dq[3] = {(uint64_t)g.D, (uint64_t)g.L, (uint64_t)g.BH};
    const uint64_t sq[2] = {(uint64_t)g.D * 2, (uint64_t)g.L * g.D * 2};
    const uint32_t bq[3] = {64, (uint32_t)kC, 1};
    const uint32_t bx[3] = {64, 64, 1};
    const uint64_t dp[3] = {(uint64_t)g.SP, (uint64_t)g.L, (uint64_t)g.BH};
    const uint64_t sp[2] = {(uint64_t)g.SP * 2, (uint64_t)g.L * g.SP * 2};
    const uint64_t deb[2] = {(uint64_t)kC, (uint64_t)nh * g.nchunks * g.RP}, seb[1] = {(uint64_t)kC * 2};
    const uint32_t beb[2] = {64, 128};
    const uint64_t dph[2] = {(uint64_t)g.R2, (uint64_t)nh * g.SP}, sph[1] = {(uint64_t)g.R2 * 2};
    const uint32_t bph[2] = {64, (uint32_t)g.SP};
    if (!make_tmap_bf16(&tq, q, 3, dq, sq, bq) || !make_tmap_bf16(&tp, a.pbuf, 3, dp, sp, bq) ||
        !make_tmap_bf16(&teb, eb, 2, deb, seb, beb) || !make_tmap_bf16(&tphi, phi, 2, dph, sph, bph))
        return cudaErrorInvalidValue;
    const int nblk = g.BH * g.G;
    if (g.G > 1) {
        // prepass uses half-chunk boxes (64 rows) for K and V
        if (!make_tmap_bf16(&tk, k, 3, dq, sq, bx) || !make_tmap_bf16(&tv, v, 3, dq, sq, bx)) return cudaErrorInvalidValue;
        const uint64_t df[2] = {(uint64_t)g.Lseg, (uint64_t)nh * g.RP}, sf[1] = {(uint64_t)g.Lseg * 2};
        const uint32_t bf[2] = {64, 128};
        if (!make_tmap_bf16(&tf, fseg, 2, df, sf, bf)) return cudaErrorInvalidValue;
        // the segment deltas, fp32 [BH][G][2][RP][D], stored by the prepass in [128 rows][32] boxes
        const uint64_t dd[2] = {(uint64_t)g.D, (uint64_t)g.BH * g.G * 2 * g.RP}, sd[1] = {(uint64_t)g.D * 4};
        const uint32_t bd[2] = {32, 128};
        if (!make_tmap_f32(&tdl, a.deltas_out, 2, dd, sd, bd)) return cudaErrorInvalidValue;
        const size_t stage_bytes = (size_t)g.NB * 128 * 64 * 2 + 2 * (size_t)64 * g.D * 2;
        const int smem = smem_request(kPreStages * stage_bytes + 256 + 1024, pow2_cols(2 * g.NB * g.D));
        if ((e = cudaFuncSetAttribute(k_prepass, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
            return e;
        {
            ProfScope ps(BLA_K_PREPASS, st);
            if ((e = launch_pdl(k_prepass, dim3(nblk), dim3(kThreads), (size_t)smem, st, tk, tv, tf, tdl, a)) !=
                cudaSuccess)
                return e;
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        long long tot = (long long)g.BH * 2 * g.M * (g.D / 4);   // k_scan: four state columns per thread
        if (tot > 0x7fffffffLL) return cudaErrorInvalidValue;        // (indexed in 32 bits)
        int blocks = (int)((tot + 255) / 256);
        if (blocks > 4096) blocks = 4096;
        {
            ProfScope ps(BLA_K_SCAN, st);
            if ((e = launch_pdl(k_scan, dim3(blocks), dim3(256), 0, st, a)) != cudaSuccess) return e;
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (!make_tmap_bf16(&tk, k, 3, dq, sq, bq) || !make_tmap_bf16(&tv, v, 3, dq, sq, bq)) return cudaErrorInvalidValue;
    {
        KLayout kl = k_layout(g);
        const int smem = smem_request(kl.total, pow2_cols(g.NB * g.D + 128 + g.RH));
        if ((e = launch_kpass(g, smem, nblk, st, tq, tk, teb, tphi, tp, a)) != cudaSuccess) return e;
    }
    {
        VLayout vl = v_layout(g);
        const int smem = smem_request(vl.total, pow2_cols(g.NB * g.D + 256));
        CUtensorMap to;
        if (!make_tmap_bf16(&to, o, 3, dq, sq, bq)) return cudaErrorInvalidValue;
        if ((e = launch_vpass(g, smem, nblk, st, tp, tv, teb, tphi, to, a)) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace bla
