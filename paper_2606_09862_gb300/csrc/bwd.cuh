// bwd.cuh -- host interface of the backward pass.
#pragma once
#include "common.cuh"

namespace bla {

// NULL if the backward supports these dimensions, else the reason it does not.
const char *bwd_unsupported(const OpDims &d);
// Workspace bytes of the backward.
size_t bwd_workspace_bytes(const OpDims &d);
// Enqueue the backward on `st`.
cudaError_t bwd_run(const OpDims &d, const void *q, const void *k, const void *v, const void *o, const void *dout,
                    const float *lse, void *dq, void *dk, void *dv, void *workspace, cudaStream_t st);

}  // namespace bla
