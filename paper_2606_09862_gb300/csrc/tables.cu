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
    size_t b = 0;
    b += align_up(sizeof(float) * (size_t)d.S * d.R2, 256);
    b += align_up(sizeof(int) * (size_t)d.S, 256);
    b += align_up(sizeof(float) * (size_t)d.M * 2, 256);
    b += align_up(sizeof(float) * (size_t)(C + 1) * d.M * 2, 256);
    return b;
}

char *tables_carve(const OpDims &d, int C, char *base, Tables *t) {
    char *p = base;
    t->phi = reinterpret_cast<float *>(p);   p += align_up(sizeof(float) * (size_t)d.S * d.R2, 256);
    t->delta = reinterpret_cast<int *>(p);   p += align_up(sizeof(int) * (size_t)d.S, 256);
    t->rot1 = reinterpret_cast<float *>(p);  p += align_up(sizeof(float) * (size_t)d.M * 2, 256);
    t->erel = reinterpret_cast<float *>(p);  p += align_up(sizeof(float) * (size_t)(C + 1) * d.M * 2, 256);
    t->C = C;
    return p;
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

cudaError_t tables_build(const OpDims &d, const Tables &t, cudaStream_t st) {
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
