// fwd_bf16.cu -- bf16 tensor-core chunked forward (placeholder until the tcgen05 kernels land).
#include "fwd_bf16.cuh"

namespace bla {

const char *fwd_bf16_unsupported(const OpDims &d) {
    (void)d;
    return "the tcgen05 chunked forward is not built yet";
}

size_t fwd_bf16_workspace_bytes(const OpDims &d) {
    (void)d;
    return 0;
}

cudaError_t fwd_bf16_run(const OpDims &d, const void *q, const void *k, const void *v, void *o, float *lse,
                         float *state_out, void *workspace, cudaStream_t st) {
    (void)d; (void)q; (void)k; (void)v; (void)o; (void)lse; (void)state_out; (void)workspace; (void)st;
    return cudaErrorNotSupported;
}

}  // namespace bla
