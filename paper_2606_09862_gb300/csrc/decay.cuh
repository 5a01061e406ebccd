// decay.cuh -- launchers of the state-decay kernels (decay.cu).
#pragma once

#include "common.cuh"

namespace bla {

// State decay (Sec. 3.3) on Alg. 1's slot-space state.  The state is fp32
// [B][H][2 (K~ then V~)][S][d]; the workspace holds the grid, the D_M table, the slot scores and,
// when lse is NULL, the log-sum-exp of the forward.
size_t decay_workspace_bytes(const OpDims &d, bool decode);
size_t decay_table_entries(const OpDims &d);   // D_M values one forward call tabulates
cudaError_t launch_decay_forward(const OpDims &d, long long pos0, const void *q, const void *k, const void *v, void *o,
                                 float *lse, const float *state_in, float *state_out, void *ws, cudaStream_t st);
cudaError_t launch_decay_decode(const OpDims &d, long long pos, const void *q, const void *k, const void *v,
                                float *state, void *o, void *ws, cudaStream_t st);
// The chunked bf16 forward and backward of the decayed form (decay_chunk.cu), for d_k = d_v in
// {64, 128} and S in {32, 64}, in 32-token chunks: tables per (head, chunk), a pass along the
// sequence for the state entering every chunk, the per-chunk work in parallel over all SMs and, in
// the backward, a reverse pass for the adjoint states.  The workspaces (decay_chunk_fwd_ws_bytes,
// decay_chunk_bwd_ws_bytes) hold the chunk states, the backward's per-chunk adjoint contributions
// (both bf16) and the tables.
bool decay_chunk_supported(const OpDims &d);
size_t decay_chunk_fwd_ws_bytes(const OpDims &d);
cudaError_t launch_decay_chunk(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                               int hs_dx, int hs_delta, const void *q, const void *k, const void *v, void *o,
                               float *lse, const float *state_in, float *state_out, void *ws, cudaStream_t st);
size_t decay_chunk_bwd_ws_bytes(const OpDims &d);
cudaError_t launch_decay_chunk_bwd(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                                   int hs_dx, int hs_delta, const void *q, const void *k, const void *v,
                                   const void *dout, const float *lse, void *dq, void *dk, void *dv, void *ws,
                                   cudaStream_t st);
// Vector-Jacobian product of the decayed forward from the zero state (dq, dk, dv in the input dtype).
size_t decay_backward_workspace_bytes(const OpDims &d);
cudaError_t launch_decay_backward(const OpDims &d, long long pos0, const void *q, const void *k, const void *v,
                                  const void *o, const void *dout, const float *lse, void *dq, void *dk, void *dv,
                                  void *ws, cudaStream_t st);

}  // namespace bla
