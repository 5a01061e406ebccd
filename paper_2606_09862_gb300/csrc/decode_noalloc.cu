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
//   * The kNoAllocScratchBytes-byte array is placed in device memory when the library's module
//     is loaded on a device: with lazy module loading (the CUDA default) that happens at the
//     first use of the module on that device, at the latest on the first call.  It stays there
//     until the process exits.  Make the first call before reserving a fixed memory budget and
//     before any stream capture.  Parameters whose tables do not fit are rejected with
//     BLA_ERR_UNSUPPORTED before anything is launched.
//   * The array's device address is looked up once per device, on the first call made with
//     that device current (cudaGetSymbolAddress), and cached for the life of the device's
//     primary context: after cudaDeviceReset the module may load elsewhere, so a process that
//     resets a device must not call this entry point on it again.
//   * All calls share the array and it keeps the previous call's contents: the tables are
//     rewritten in full by every call, so nothing needs clearing, but two calls that overlap
//     on the GPU (different streams without ordering) race on it.
#include <math.h>
#include <stdio.h>

#include <atomic>

#include "common.cuh"

namespace bla {

namespace {

constexpr size_t kNoAllocScratchBytes = 512 * 1024;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

// Device address of g_decode_scratch for the current device (looked up once per device; host
// threads that race on the first lookup store the same value).
cudaError_t scratch_address(void **out) {
    static std::atomic<void *> addr[kMaxDevices];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    void *p = addr[dev].load(std::memory_order_acquire);
    if (!p) {
        e = cudaGetSymbolAddress(&p, g_decode_scratch);
        if (e != cudaSuccess) return e;
        addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
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
    NvtxRange nvtx("bla_decode_step_noalloc");
    OpDims d;
    const bla_status s = check_decode(p, pos, q, k, v, state, o, &d);
    if (s != BLA_OK) return s;
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
