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
// The chunked bf16 forward of the decayed form (decay_chunk.cu): 64-token chunks with the
// contractions on the tensor cores, for d_k = d_v in {64, 128} and S in {32, 64}.  Each head's
// sequence runs as G segments of cps chunks (state deltas, a scan, then the outputs).
struct DcPlan {
    int G, cps;
};
bool decay_chunk_supported(const OpDims &d);
DcPlan decay_chunk_plan(const OpDims &d);
cudaError_t launch_decay_chunk(const OpDims &d, long long pos0, int dmax, const float *Dx, const int *delta,
                               int hs_dx, int hs_delta, const void *q, const void *k, const void *v, void *o,
                               float *lse, const float *state_in, float *state_out, float *seg_delta,
                               float *seg_decay, float *win, cudaStream_t st);
// Its backward (decay_chunk_bwd.cu), for the same shapes, in 32-token chunks: tables, a pass for the
// state entering every chunk, the per-chunk chains in parallel, and a reverse pass for the adjoint
// states; the workspace (decay_chunk_bwd_ws_bytes) holds the chunk states, the chunks' adjoint
// contributions (both bf16) and the tables.
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
