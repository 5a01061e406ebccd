// decode_noalloc.cu -- bla_decode_step_noalloc: the decode step for callers that may not
// allocate device memory.
//
// The regular bla_decode_step takes a caller-provided workspace for its interpolation and
// phase tables.  Some callers cannot provide one: an inference server plugin that runs
// inside a fixed, pre-reserved memory budget, or a latency-critical token loop where the
// host must not call cudaMalloc (it can synchronise the device and stall every other
// stream).  This variant keeps the tables in a fixed device array that belongs to the
// library module, so the call itself allocates nothing.
//
//   * kNoAllocScratchBytes bytes of device memory are reserved per GPU that loads the
//     library, for the lifetime of the process.  Parameters whose tables do not fit are
//     rejected with BLA_ERR_UNSUPPORTED before anything is launched.
//   * The array's device address is looked up once per device, on the first call made with
//     that device current (cudaGetSymbolAddress); make that first call before any stream
//     capture.  Later calls on the same device reuse the address.
//   * All calls share the array and it keeps the previous call's contents: the tables are
//     rewritten in full by every call, so nothing needs clearing, but two calls that overlap
//     on the GPU (different streams without ordering) race on it.
#include <math.h>
#include <stdio.h>

#include "common.cuh"

namespace bla {

namespace {

constexpr size_t kNoAllocScratchBytes = 512 * 1024;
constexpr int kMaxDevices = 64;
constexpr double kPi = 3.14159265358979323846;

static __device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

// Device address of g_decode_scratch for the current device (looked up once per device).
cudaError_t scratch_address(void **out) {
    static void *addr[kMaxDevices] = {nullptr};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (!addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_decode_scratch);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *out = addr[dev];
    return cudaSuccess;
}

bla_status reject(bla_status s, const char *fmt, long long a = 0, long long b = 0) {
    char buf[256];
    snprintf(buf, sizeof(buf), fmt, a, b);
    set_last_error(buf);
    return s;
}

}  // namespace

}  // namespace bla

using namespace bla;

extern "C" bla_status bla_decode_step_noalloc(const bla_params *p, long long pos, const void *q, const void *k,
                                              const void *v, float *state, void *o, void *stream) {
    set_last_error("");
    if (!p) return reject(BLA_ERR_INVALID, "params is NULL");
    if (p->B < 1 || p->H < 1 || p->M < 1 || p->d_k < 1 || p->d_v < 1)
        return reject(BLA_ERR_INVALID, "B, H, M, d_k and d_v must be >= 1");
    if (!(p->window > 0.0) || !isfinite(p->window) || !isfinite(p->omega) || !isfinite(p->scale))
        return reject(BLA_ERR_INVALID, "window must be > 0; omega and scale finite");
    if (p->dtype != BLA_F32 && p->dtype != BLA_BF16) return reject(BLA_ERR_INVALID, "dtype must be BLA_F32 or BLA_BF16");
    const double Te = fmax(p->window, 2.0 * p->M - 1.0);
    if (p->S < 1 || (double)p->S > Te) return reject(BLA_ERR_INVALID, "S must be in [1, T] (S=%lld)", p->S);
    if (pos < 0) return reject(BLA_ERR_INVALID, "pos must be >= 0 (got %lld)", pos);
    if (p->periods) return reject(BLA_ERR_UNSUPPORTED, "the no-alloc decode does not support per-head periods yet");
    if (!q || !k || !v || !state || !o) return reject(BLA_ERR_INVALID, "q, k, v, state and o must be non-NULL");
    const uintptr_t mis = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) |
                          reinterpret_cast<uintptr_t>(v) | reinterpret_cast<uintptr_t>(state) |
                          reinterpret_cast<uintptr_t>(o);
    if (mis & 15u) return reject(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if (p->d_k != p->d_v || (p->d_k != 32 && p->d_k != 64 && p->d_k != 128))
        return reject(BLA_ERR_UNSUPPORTED, "decode needs d_k = d_v in {32, 64, 128} (got %lld, %lld)", p->d_k, p->d_v);
    if (p->S > 256) return reject(BLA_ERR_UNSUPPORTED, "decode needs S <= 256 (got %lld)", p->S);
    if (p->phase_mode != BLA_PHASE_LAG && p->phase_mode != BLA_PHASE_ABSOLUTE)
        return reject(BLA_ERR_INVALID, "phase_mode must be BLA_PHASE_LAG or BLA_PHASE_ABSOLUTE (got %lld)",
                      (long long)p->phase_mode);
    OpDims d;
    d.B = p->B; d.H = p->H; d.L = 1; d.dk = p->d_k; d.dv = p->d_v; d.M = p->M; d.S = p->S; d.R2 = 2 * p->M;
    d.T = Te;
    d.w = p->omega > 0.0 ? p->omega : 2.0 * kPi / Te;
    d.scale = (float)(p->scale > 0.0 ? p->scale : 1.0 / sqrt((double)p->d_k));
    d.dtype = p->dtype;
    d.absolute = p->phase_mode == BLA_PHASE_ABSOLUTE;
    d.periods = nullptr;
    d.omega_in = p->omega;
    const size_t need = tables_bytes(d, 0);
    if (need > kNoAllocScratchBytes)
        return reject(BLA_ERR_UNSUPPORTED,
                      "tables need %lld bytes, more than the %lld-byte static scratch of the no-alloc decode",
                      (long long)need, (long long)kNoAllocScratchBytes);
    void *scratch = nullptr;
    cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess) {
        set_last_error(cudaGetErrorString(e));
        return BLA_ERR_CUDA;
    }
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Tables t;
    tables_carve(d, 0, static_cast<char *>(scratch), &t);
    e = tables_build(d, t, st);
    if (e == cudaSuccess) e = launch_decode(d, pos, t, q, k, v, state, o, st);
    if (e != cudaSuccess) {
        set_last_error(cudaGetErrorString(e));
        return BLA_ERR_CUDA;
    }
    return BLA_OK;
}
