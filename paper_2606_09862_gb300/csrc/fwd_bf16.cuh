// fwd_bf16.cuh -- host interface of the bf16 tensor-core chunked forward.
#pragma once
#include "common.cuh"

namespace bla {

// NULL if the bf16 forward supports these dimensions, else the reason it does not.
const char *fwd_bf16_unsupported(const OpDims &d);
// Workspace bytes of the bf16 forward (tables, segment states, inter-pass buffers).
size_t fwd_bf16_workspace_bytes(const OpDims &d);
// Build the bf16 operand tables EB [RP][128] and PHI [SP][2M] (no segment table).
cudaError_t build_bf16_tables(const OpDims &d, int RP, int SP, __nv_bfloat16 *eb, __nv_bfloat16 *phi, cudaStream_t st);
// Enqueue the bf16 forward on `st`.
cudaError_t fwd_bf16_run(const OpDims &d, const void *q, const void *k, const void *v, void *o, float *lse,
                         float *state_out, void *workspace, cudaStream_t st);

}  // namespace bla
