// tables.cu -- device-side construction of the interpolation and phase tables.
//
// Everything is evaluated in fp64 from integer indices and rounded once to fp32:
//   dilated lags   D_j = round(j T / S)       (Alg. 1-3 "dilated_time", generalised to S slots;
//                                              round half to even)
//   coefficients   A[j,m] = c_m cos(m w D_j), B[j,m] = c_m sin(m w D_j), c_0 = 1/(2M-1),
//                  c_{m>0} = 2/(2M-1)          (Eq. translated); B is negated for the
//                  absolute form (Alg. 1), whose slots read e^{+i m w D_j}
//   one-step rotation cos(m w), sin(m w)       (Eq. recurrence)
//   chunk phases   cos(m w tau), sin(m w tau), tau = 0..C
#include "common.cuh"

namespace bla {

size_t tables_bytes(const OpDims &d, int C) {
    const size_t nh = d.periods ? (size_t)d.H : 1;
    size_t b = 0;
    b += align_up(sizeof(float) * nh * d.S * d.R2, 256);
    b += align_up(sizeof(int) * nh * d.S, 256);
    b += align_up(sizeof(float) * nh * d.M * 2, 256);
    b += align_up(sizeof(float) * nh * (C + 1) * d.M * 2, 256);
    if (d.periods) b += align_up(sizeof(double) * nh, 256);
    return b;
}

char *tables_carve(const OpDims &d, int C, char *base, Tables *t) {
    const size_t nh = d.periods ? (size_t)d.H : 1;
    char *p = base;
    t->phi = reinterpret_cast<float *>(p);   p += align_up(sizeof(float) * nh * d.S * d.R2, 256);
    t->delta = reinterpret_cast<int *>(p);   p += align_up(sizeof(int) * nh * d.S, 256);
    t->rot1 = reinterpret_cast<float *>(p);  p += align_up(sizeof(float) * nh * d.M * 2, 256);
    t->erel = reinterpret_cast<float *>(p);  p += align_up(sizeof(float) * nh * (C + 1) * d.M * 2, 256);
    t->wh = nullptr;
    if (d.periods) {
        t->wh = reinterpret_cast<double *>(p);
        p += align_up(sizeof(double) * nh, 256);
    }
    const int per = d.periods ? 1 : 0;
    t->hs_phi = per * d.S * d.R2;
    t->hs_delta = per * d.S;
    t->hs_rot1 = per * d.M * 2;
    t->hs_erel = per * (C + 1) * d.M * 2;
    t->C = C;
    return p;
}

void head_periods(const OpDims &d, double omega, HeadPeriods *hp) {
    const double pi = 3.14159265358979323846;
    const double floor_T = 2.0 * d.M - 1.0;
    hp->n = d.periods ? d.H : 0;
    for (int h = 0; h < hp->n; ++h) {
        const double T = d.periods[h] < floor_T ? floor_T : d.periods[h];
        hp->T[h] = T;
        hp->w[h] = omega > 0.0 ? omega : 2.0 * pi / T;
    }
}

__global__ void k_tables(int M, int S, double T, double w, int C, float sin_sign, float *phi, int *delta,
                         float *rot1, float *erel) {
    const int R2 = 2 * M;
    const double n = 2.0 * M - 1.0;
    const long long n_phi = (long long)S * R2;
    const long long n_rot = (long long)M;
    const long long n_erel = (long long)(C + 1) * M;
    const long long total = n_phi + S + n_rot + n_erel;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        if (i < n_phi) {
            int j = (int)(i / R2), r = (int)(i % R2), m = r >> 1;
            double dj = rint((double)j * T / (double)S);
            double c = (m == 0) ? 1.0 / n : 2.0 / n;
            double ang = (double)m * w * dj;
            phi[i] = (float)(c * ((r & 1) ? sin_sign * sin(ang) : cos(ang)));
        } else if (i < n_phi + S) {
            int j = (int)(i - n_phi);
            delta[j] = (int)rint((double)j * T / (double)S);
        } else if (i < n_phi + S + n_rot) {
            int m = (int)(i - n_phi - S);
            double s, c;
            sincos((double)m * w, &s, &c);
            rot1[2 * m] = (float)c;
            rot1[2 * m + 1] = (float)s;
        } else {
            long long e = i - n_phi - S - n_rot;
            int tau = (int)(e / M), m = (int)(e % M);
            double s, c;
            sincos((double)m * w * (double)tau, &s, &c);
            erel[2 * e] = (float)c;
            erel[2 * e + 1] = (float)s;
        }
    }
}

// The same tables for every head h < hp.n at its own period: element i of head h goes to the
// head's slice (strides hs_*), and wh[h] = w_h.
__global__ void k_tables_heads(HeadPeriods hp, int M, int S, int C, float sin_sign, Tables t) {
    const long long per = (long long)S * 2 * M + S + M + (long long)(C + 1) * M + 1;
    const long long total = per * hp.n;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int h = (int)(i / per);
        long long e = i % per;
        const double T = hp.T[h], w = hp.w[h];
        const int R2 = 2 * M;
        const double n = 2.0 * M - 1.0;
        if (e < (long long)S * R2) {
            const int j = (int)(e / R2), r = (int)(e % R2), m = r >> 1;
            const double dj = rint((double)j * T / (double)S);
            const double c = (m == 0) ? 1.0 / n : 2.0 / n;
            const double ang = (double)m * w * dj;
            t.phi[(size_t)h * t.hs_phi + e] = (float)(c * ((r & 1) ? sin_sign * sin(ang) : cos(ang)));
            continue;
        }
        e -= (long long)S * R2;
        if (e < S) {
            t.delta[(size_t)h * t.hs_delta + e] = (int)rint((double)e * T / (double)S);
            continue;
        }
        e -= S;
        if (e < M) {
            double sn, cs;
            sincos((double)e * w, &sn, &cs);
            t.rot1[(size_t)h * t.hs_rot1 + 2 * e] = (float)cs;
            t.rot1[(size_t)h * t.hs_rot1 + 2 * e + 1] = (float)sn;
            continue;
        }
        e -= M;
        if (e < (long long)(C + 1) * M) {
            const int tau = (int)(e / M), m = (int)(e % M);
            double sn, cs;
            sincos((double)m * w * (double)tau, &sn, &cs);
            t.erel[(size_t)h * t.hs_erel + 2 * e] = (float)cs;
            t.erel[(size_t)h * t.hs_erel + 2 * e + 1] = (float)sn;
            continue;
        }
        t.wh[h] = w;
    }
}

cudaError_t tables_build_heads(const OpDims &d, double omega, const Tables &t, cudaStream_t st) {
    HeadPeriods hp;
    head_periods(d, omega, &hp);
    const long long total = ((long long)d.S * d.R2 + d.S + d.M + (long long)(t.C + 1) * d.M + 1) * hp.n;
    int blocks = (int)((total + 255) / 256);
    if (blocks > 1024) blocks = 1024;
    ProfScope ps(BLA_K_TABLES, st);
    k_tables_heads<<<blocks, 256, 0, st>>>(hp, d.M, d.S, t.C, d.absolute ? -1.f : 1.f, t);
    return cudaGetLastError();
}

cudaError_t tables_build(const OpDims &d, const Tables &t, cudaStream_t st) {
    if (d.periods) return tables_build_heads(d, d.omega_in, t, st);
    long long total = (long long)d.S * d.R2 + d.S + d.M + (long long)(t.C + 1) * d.M;
    int threads = 256;
    int blocks = (int)((total + threads - 1) / threads);
    if (blocks > 1024) blocks = 1024;
    ProfScope ps(BLA_K_TABLES, st);
    k_tables<<<blocks, threads, 0, st>>>(d.M, d.S, d.T, d.w, t.C, d.absolute ? -1.f : 1.f, t.phi, t.delta, t.rot1,
                                         t.erel);
    return cudaGetLastError();
}

}  // namespace bla
