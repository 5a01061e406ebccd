// common.cuh -- shared definitions of the BLA CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/bla.h"

namespace bla {

// Error codes written to the device error word by bounded waits.
enum : int {
    DEVERR_NONE = 0,
    DEVERR_MBAR_TIMEOUT = 1,   // an mbarrier wait exceeded its poll budget
    DEVERR_SMEM_ALIGN = 2,     // a kernel found its dynamic shared memory base misaligned
};

// Derived operator constants (host side), from bla_params.
struct OpDims {
    int B, H, L, dk, dv, M, S, R2;   // R2 = 2M interleaved state rows (cos m, sin m)
    double T;                        // clamped period
    double w;                        // mode frequency omega
    float scale;
    int dtype;
    int absolute;                    // 1: absolute-phase slots (Alg. 1), 0: lag form (Alg. 2)
    const double *periods;           // host array of H per-head periods (raw, before the clamp), or
                                     // NULL when every head uses T; never read on the device
    double omega_in;                 // the caller's omega (> 0: the frequency of every head)
};

// Per-head periods handed to the table builders by value (Alg. 1 and Alg. 3: T in R^H).
constexpr int kMaxHeadPeriods = 256;
struct HeadPeriods {
    int n;
    double T[kMaxHeadPeriods];   // clamped periods
    double w[kMaxHeadPeriods];   // mode frequencies
};
// Fill `hp` from d.periods (clamp to 2M-1; omega > 0 overrides every head's 2 pi / T_h).
void head_periods(const OpDims &d, double omega, HeadPeriods *hp);

// Table block (built on the device per call; lives in the caller's workspace).
//   phi   [S][R2] fp32: phi[j][2m] = c_m cos(m w D_j), phi[j][2m+1] = sigma c_m sin(m w D_j)
//         with c_0 = 1/(2M-1), c_m = 2/(2M-1) (Eq. translated); sigma = +1 in the lag form,
//         -1 in the absolute form (its slots read e^{+i m w D_j} where the lag form reads
//         e^{-i m w D_j}).
//   delta [S] int: dilated lags round(j T / S).
//   rot1  [M][2] fp32: cos(m w), sin(m w) (Eq. recurrence, one step).
//   erel  [C+1][M][2] fp32: cos(m w tau), sin(m w tau), tau = 0..C (chunk phases).
//   With per-head periods each table is repeated per head; hs_* are the per-head element strides
//   (0 when the heads share one period) and wh[H] holds each head's mode frequency (NULL when shared:
//   kernels then use OpDims::w).
struct Tables {
    float *phi;
    int *delta;
    float *rot1;
    float *erel;
    int C;
    int hs_phi, hs_delta, hs_rot1, hs_erel;
    double *wh;
};

// Point `t` at head h's tables; returns head h's mode frequency.
__device__ __forceinline__ double tables_for_head(Tables &t, int h, double w_shared) {
    t.phi += (size_t)h * t.hs_phi;
    t.delta += (size_t)h * t.hs_delta;
    t.rot1 += (size_t)h * t.hs_rot1;
    t.erel += (size_t)h * t.hs_erel;
    return t.wh ? t.wh[h] : w_shared;
}

// Bytes taken by the table block for a given chunk length (each part 256-aligned).
size_t tables_bytes(const OpDims &d, int C);
// Carve the table block out of `base` (256-aligned) and return the next free byte.
char *tables_carve(const OpDims &d, int C, char *base, Tables *t);
// Launch the table builder (fp64 arithmetic, rounded to fp32).
cudaError_t tables_build(const OpDims &d, const Tables &t, cudaStream_t st);

static inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

__device__ __forceinline__ float bf16_to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ float load_elem(const T *p, size_t i);
template <> __device__ __forceinline__ float load_elem<float>(const float *p, size_t i) { return p[i]; }
template <> __device__ __forceinline__ float load_elem<__nv_bfloat16>(const __nv_bfloat16 *p, size_t i) {
    return __bfloat162float(p[i]);
}
template <typename T> __device__ __forceinline__ void store_elem(T *p, size_t i, float x);
template <> __device__ __forceinline__ void store_elem<float>(float *p, size_t i, float x) { p[i] = x; }
template <> __device__ __forceinline__ void store_elem<__nv_bfloat16>(__nv_bfloat16 *p, size_t i, float x) {
    p[i] = __float2bfloat16_rn(x);
}

// Replace the calling thread's bla_last_error_string() text.
void set_last_error(const char *msg);

// Device address of the library's error word (a __device__ int of this module, one per
// device); kernels with bounded waits receive it as an argument.  NULL on failure.
int *device_error_word();

__device__ __forceinline__ void report_device_error(int *word, int code) {
    if (word) atomicCAS(word, 0, code);
}

// Launch accounting and optional per-launch event timing (api.cu).  Construct a ProfScope
// immediately before a kernel launch and let it go out of scope right after it.
struct ProfScope {
    ProfScope(int kernel_id, cudaStream_t st);
    ~ProfScope();
    int kid;
    cudaStream_t stream;
    int slot;
};

// Launch `kernel` so that it may start while the previous kernel in the stream finishes
// (programmatic stream serialization): the kernel must call tc::pdl_wait() before it reads
// anything the previous kernels wrote, and write nothing before that.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// Launchers of the individual kernels (defined in their .cu files).
cudaError_t launch_forward_f32(const OpDims &d, int C, const Tables &t, const float *q, const float *k,
                               const float *v, float *o, float *lse, float *state_out, float *scratch,
                               cudaStream_t st);
size_t forward_f32_scratch_bytes(const OpDims &d, int C);
int forward_f32_smem_bytes(const OpDims &d, int C);

cudaError_t launch_decode(const OpDims &d, long long pos, const Tables &t, const void *q, const void *k,
                          const void *v, float *state, void *o, cudaStream_t st);
// Dynamic shared memory of one decode launch (the launcher opts in above 48 KB).
int decode_smem_bytes(const OpDims &d);

// Checks shared by both decode entry points (api.cu): the common parameter checks, pos >= 0,
// non-NULL 16-byte-aligned tensors, d_k = d_v in {32, 64, 128}, S <= 256 and the decode's shared
// memory; fills `d`.  Sets the thread's last-error text on failure.
bla_status check_decode(const bla_params *p, long long pos, const void *q, const void *k, const void *v,
                        const float *state, const void *o, OpDims *d);

// An NVTX range around an entry point (visible in Nsight timelines; free when no tool listens).
struct NvtxRange {
    explicit NvtxRange(const char *name);
    ~NvtxRange();
};

}  // namespace bla
