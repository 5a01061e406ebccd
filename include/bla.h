/*
 * bla.h -- C ABI of the GB300 (sm_103a) Blurry Window Attention library, libbla_gb300.so.
 *
 * The operator (arxiv 2606.09862, "Blurry Window Attention", Sec. 3.1):
 * per batch element b and head h, keys and values are written into a finite
 * frequency window of M Fourier modes, a rotating state advanced by e^{i m w}
 * (Eq. recurrence):
 *     Kcos[m] <- cos(m w) Kcos[m] - sin(m w) Ksin[m] + k_t
 *     Ksin[m] <- sin(m w) Kcos[m] + cos(m w) Ksin[m]          (V likewise)
 * S blurry slots are rebuilt from the state with the translated Dirichlet
 * coefficients A, B of Eq. (translated) at the dilated lags Delta_j (Eq. compressed),
 *     K~[j] = sum_m A[j,m] Kcos[m] + B[j,m] Ksin[m],
 * and the query attends over the slots with a softmax whose mask hides slots
 * before the start of the sequence, t >= Delta_j (Eq. output; Alg. 2):
 *     o_t = softmax_j(scale * q_t . K~[j] + mask) . V~.
 *
 * Conventions shared by every entry point
 *   - All tensor arguments are DEVICE pointers owned by the caller; the library
 *     allocates no device memory.  Scratch memory, where needed, is the
 *     caller's `workspace` of at least bla_workspace_bytes() bytes, 256-byte
 *     aligned.  Tensor pointers must be 16-byte aligned.
 *   - q, k: [B][H][L][d_k]; v, o, dout: [B][H][L][d_v]; contiguous, element type
 *     `dtype` (fp32 or bf16).  lse: [B][H][L] fp32 (natural-log log-sum-exp of the
 *     unmasked slot scores).
 *   - Recurrent state: fp32 [B][H][2 (K then V)][M][2 (cos, sin)][d], d = d_k for
 *     the K half and d_v for the V half.  Row (m, sin) at m = 0 is the sine of the
 *     zero frequency: it is always 0 and is neither read nor written.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Every call is
 *     asynchronous on that stream; argument errors are detected on the host
 *     before any launch.
 *   - Nothing is thrown across the ABI; every function returns a bla_status.
 *     bla_last_error_string() describes the most recent failure of the calling
 *     thread.
 *   - Bounded device waits: every wait inside a kernel gives up after a fixed
 *     number of polls, records a code in the library's device error word and
 *     returns.  bla_device_error() synchronises the stream and reports it as
 *     BLA_ERR_TIMEOUT.
 */
#ifndef BLA_GB300_H
#define BLA_GB300_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BLA_OK = 0,
    BLA_ERR_INVALID = 1,      /* bad argument (null pointer, size, alignment, range) */
    BLA_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels implement */
    BLA_ERR_CUDA = 3,         /* a CUDA runtime/driver call or a launch failed */
    BLA_ERR_TIMEOUT = 4       /* a bounded device wait gave up (see bla_device_error) */
} bla_status;

typedef enum { BLA_F32 = 0, BLA_BF16 = 1 } bla_dtype;

/* Operator parameters (Alg. 1-3 inputs: Q, K, V, period T, interpolation
 * matrices A, B built from M, S and T, chunk size C). */
typedef struct {
    int B, H, L;        /* batch, heads, sequence length (L ignored by bla_decode_step) */
    int d_k, d_v;       /* head dimensions */
    int M;              /* Fourier modes, m = 0..M-1; 2M-1 live state rows per K and V */
    int S;              /* slots; 1 <= S <= T.  The paper uses S = 2M-1 */
    double window;      /* period T (> 0); clamped to max(T, 2M-1) as in Alg. 1 and 3 */
    double omega;       /* <= 0: 2*pi/T (Sec. 3.1); > 0: used as the mode frequency w */
    int chunk;          /* chunk length C of the fp32 path; 0 = default (64).  The bf16
                           path always tiles by 128 tokens.  Results do not depend on it
                           beyond rounding. */
    double scale;       /* softmax scale; <= 0: 1/sqrt(d_k) (Eq. output, per head) */
    int dtype;          /* bla_dtype of q, k, v, o, dout, dq, dk, dv */
    int phase_mode;     /* bla_phase_mode: how the slots index time (0 = the lag form) */
    const double *periods;  /* NULL: every head uses `window`.  Else a HOST array of H periods, one
                               per head (Alg. 1 and Alg. 3 take T in R^H): head h's grid, frequency
                               (2*pi/T_h unless omega > 0) and coefficients follow periods[h], each
                               clamped to max(T_h, 2M-1); S must not exceed any of them.  Read
                               during the call only.  At most 256 heads.  Supported by every
                               entry point; bla_backward then runs the (batch, head) slices one
                               after the other, each at its own period. */
} bla_params;

/* How a slot reads the past (bla_params.phase_mode).
 *   BLA_PHASE_LAG       the recurrent definition (Eq. recurrence, Eq. compressed, Alg. 2):
 *                       slot j of token t weights key u by D_M(t - u - Delta_j), a window
 *                       at lag Delta_j behind t.
 *   BLA_PHASE_ABSOLUTE  the time-rolling form the paper runs in practice (Sec. 3.2, Alg. 1,
 *                       Alg. 3): slot j weights key u by D_M(u - Delta_j), a kernel anchored
 *                       at absolute phase Delta_j (mod T).  The two agree only when
 *                       T = S = 2M-1.
 * D_M is the translated Dirichlet kernel of Eq. (translated); the slot mask (keep slot j
 * of token t iff t >= Delta_j) and the state (the lag-frame mode state of Eq. recurrence,
 * so a prefill hands over to decode identically) are the same in both modes. */
typedef enum { BLA_PHASE_LAG = 0, BLA_PHASE_ABSOLUTE = 1 } bla_phase_mode;

/* Which entry point a workspace size is asked for. */
typedef enum {
    BLA_WS_FORWARD = 0, BLA_WS_BACKWARD = 1, BLA_WS_DECODE = 2, BLA_WS_FORWARD_HOST = 3,
    BLA_WS_DECAY_FORWARD = 4, BLA_WS_DECAY_DECODE = 5, BLA_WS_DECAY_BACKWARD = 6
} bla_ws_kind;

/*
 * Bytes of device workspace the entry point `which` (a bla_ws_kind) needs for
 * these parameters.  The workspace holds the interpolation tables (built on the
 * device at every call) and, for the chunked paths, per-segment states and
 * inter-pass intermediates.  Returns 0 for invalid parameters; call the entry
 * point to get the error.
 */
size_t bla_workspace_bytes(const bla_params *p, int which);

/*
 * Chunked forward (prefill) over L tokens from the zero state (Sec. 3.1: "These
 * states are initialized to zero"; Alg. 3 chunk form, computed in the lag frame of
 * Eq. recurrence).
 *   q, k, v    inputs as described above (device).
 *   o          output [B][H][L][d_v] (device), dtype of the inputs.
 *   lse        optional [B][H][L] fp32 (device) or NULL; needed by bla_backward.
 *   state_out  optional fp32 state after the last token (device) or NULL; it is
 *              the state bla_decode_step continues from with pos = L.
 *   workspace  device scratch of >= bla_workspace_bytes(p, BLA_WS_FORWARD) bytes.
 * dtype BLA_F32: fp32 SIMT path.  dtype BLA_BF16: tcgen05 tensor-core path with
 * bf16 operands and fp32 accumulation; requires d_k = d_v in {64, 128},
 * 2M in {64, 128, 256} and S in {32, 64, 128} (else BLA_ERR_UNSUPPORTED).
 */
bla_status bla_forward_chunked(const bla_params *p, const void *q, const void *k, const void *v,
                               void *o, float *lse, float *state_out,
                               void *workspace, size_t ws_bytes, void *stream);

/*
 * bla_forward_chunked on tensors in HOST memory (no paper counterpart: a serving convenience).
 * q, k, v are read from and o is written to host memory, in the layout of bla_forward_chunked.
 * The B*H heads are independent, so they are processed in groups: each group's host-to-device
 * copies, its forward and its device-to-host copy run on separate streams (two owned by the
 * library, created on first use on each device), and copies overlap the other groups' compute.
 *   - The host buffers should be page-locked (cudaHostAlloc or cudaHostRegister); pageable
 *     memory gives the same results without the overlap.
 *   - workspace: device scratch of >= bla_workspace_bytes(p, BLA_WS_FORWARD_HOST) bytes; it holds
 *     the device copies of q, k, v and o and the forward's own workspace.
 *   - The call returns once everything is enqueued.  o is complete on the host once `stream` has
 *     been synchronised (the stream waits for the last copy); the host buffers must stay valid and
 *     untouched until then.  Calls must be ordered by the caller (they share the library's streams
 *     and the caller's workspace).
 * Results equal bla_forward_chunked's to rounding (the heads of a group are one launch, so the
 * sequence segmentation may differ).  lse and the final state are not returned.
 */
bla_status bla_forward_chunked_host(const bla_params *p, const void *q, const void *k, const void *v, void *o,
                                    void *workspace, size_t ws_bytes, void *stream);

/*
 * One single-token decode step for B*H independent sequences (Alg. 2 loop body).
 *   pos        0-based absolute index of this token in its sequence (>= 0); the
 *              slot mask keeps slot j iff pos >= Delta_j.
 *   q, k, v    [B][H][d_k] / [B][H][d_k] / [B][H][d_v] (device), dtype p->dtype.
 *   state      fp32 state (device), read and updated in place: on return it
 *              includes this token.
 *   o          [B][H][d_v] (device), dtype p->dtype.
 *   workspace  device scratch of >= bla_workspace_bytes(p, BLA_WS_DECODE) bytes.
 * p->L is ignored.  Requires d_k = d_v in {32, 64, 128}, S <= 256, and
 * 4 (2M + S + 8 d_k) bytes of shared memory at most 227 KB (M up to about 28,000);
 * other sizes return BLA_ERR_UNSUPPORTED before any launch.
 */
bla_status bla_decode_step(const bla_params *p, long long pos, const void *q, const void *k,
                           const void *v, float *state, void *o, void *workspace, size_t ws_bytes,
                           void *stream);

/*
 * bla_decode_step for callers that may not allocate device memory (the paper has no
 * counterpart; this is a deployment convenience).  Same arguments and results as
 * bla_decode_step, without the workspace: the step's tables live in a fixed 512 KiB
 * device array owned by the library.  Meant for callers that run within a fixed,
 * pre-reserved memory budget or must not call the allocator mid-step (cudaMalloc can
 * synchronise the device).
 *   - The array takes its 512 KiB of device memory when the library's module is loaded
 *     on a device (with lazy module loading, the CUDA default, at the first use of the
 *     module there, at the latest on the first call) and keeps it until exit.  Make the
 *     first call before reserving a fixed memory budget and before any stream capture.
 *   - Parameters whose tables exceed the array are rejected with BLA_ERR_UNSUPPORTED
 *     before any launch; the argument checks are those of bla_decode_step.
 *   - The array's device address is looked up on the first call made on each device and
 *     kept for the life of that device's primary context: do not call this entry point
 *     on a device after cudaDeviceReset.
 *   - All calls share the array (it keeps the last call's tables, rewritten in full by
 *     every call): calls that overlap on the GPU race and must be ordered by the caller.
 */
bla_status bla_decode_step_noalloc(const bla_params *p, long long pos, const void *q, const void *k,
                                   const void *v, float *state, void *o, void *stream);

/*
 * Backward pass of bla_forward_chunked: given dout = dL/do, writes dq, dk, dv
 * (same shapes and dtype as q, k, v).  o and lse are the forward's outputs.
 * The vector-Jacobian product of the operator defined by Eqs. (recurrence),
 * (compressed) and (output); the paper trains through it but prints no formula.
 */
bla_status bla_backward(const bla_params *p, const void *q, const void *k, const void *v,
                        const void *o, const void *dout, const float *lse,
                        void *dq, void *dk, void *dv, void *workspace, size_t ws_bytes, void *stream);

/* ---------------------------------------------------------------- state decay (Sec. 3.3)
 * Alg. 1 (the absolute form) with the decay of Sec. 3.3.  The state is Alg. 1's slot-space state,
 * fp32 [B][H][2 (K~ then V~)][S][d], and token t (absolute index) updates every slot j as
 *     K~[j] <- (1 - D_j(t)) K~[j] + D_j(t) k_t,      V~[j] likewise,
 * with D_j(t) = D_M(t - Delta_j) the weight Alg. 1 adds the token with ("interpolate", Eq.
 * compressed_simplified); then o_t = softmax_j(scale q_t . K~[j], slots with t >= Delta_j) . V~.
 * At T = 2M-1 the decay keeps in slot j the latest token t = Delta_j (mod 2M-1), which at S = 2M-1
 * is sliding-window attention over the last 2M-1 tokens.  Shared requirements: phase_mode =
 * BLA_PHASE_ABSOLUTE (the decay is defined on that form's slots; BLA_PHASE_LAG returns
 * BLA_ERR_UNSUPPORTED), d_k = d_v in {32, 64, 128} and S <= 256 (else BLA_ERR_UNSUPPORTED). */

/*
 * Forward over L tokens, continuing from `state_in` (NULL = zero state) at absolute index pos0
 * (>= 0; it sets the phase of D_j and the slot mask; 0 for a fresh sequence).
 *   o          [B][H][L][d_v] (device), dtype of the inputs.
 *   lse        optional [B][H][L] fp32 (device) or NULL.
 *   state_in   optional slot-space state (device) the tokens continue from, or NULL.
 *   state_out  optional slot-space state after the last token (device), or NULL; it may be the
 *              same pointer as state_in (updated in place) but must not overlap it otherwise.
 *   workspace  device scratch of >= bla_workspace_bytes(p, BLA_WS_DECAY_FORWARD) bytes (it holds
 *              the B*H*S*L fp32 slot scores and a table of L + T values of D_M).
 * dtype BLA_F32 or BLA_BF16 (fp32 state and arithmetic either way).  A period with L + T above
 * 2^30 returns BLA_ERR_UNSUPPORTED.
 */
bla_status bla_decay_forward(const bla_params *p, long long pos0, const void *q, const void *k, const void *v,
                             void *o, float *lse, const float *state_in, float *state_out, void *workspace,
                             size_t ws_bytes, void *stream);

/*
 * One decode step of the decayed form for B*H sequences at absolute index pos (>= 0).
 *   q, k, v    [B][H][d_k] / [B][H][d_k] / [B][H][d_v] (device), dtype p->dtype.
 *   state      slot-space state (device), read and updated in place.
 *   o          [B][H][d_v] (device).
 *   workspace  device scratch of >= bla_workspace_bytes(p, BLA_WS_DECAY_DECODE) bytes.
 * p->L is ignored.  A prefill of L tokens by bla_decay_forward hands over with pos = L.
 */
bla_status bla_decay_decode_step(const bla_params *p, long long pos, const void *q, const void *k, const void *v,
                                 float *state, void *o, void *workspace, size_t ws_bytes, void *stream);

/*
 * Backward of bla_decay_forward from the zero state (state_in = NULL), tokens at absolute indices
 * pos0 ..: given dout = dL/do, writes dq, dk, dv (shapes and dtype of q, k, v).  o and lse are the
 * forward's outputs.  The vector-Jacobian product of the decayed recurrence; the paper trains
 * through it but prints no formula.
 *   workspace  device scratch of >= bla_workspace_bytes(p, BLA_WS_DECAY_BACKWARD) bytes (two
 *              B*H*S*L fp32 buffers and the D_M table).
 */
bla_status bla_decay_backward(const bla_params *p, long long pos0, const void *q, const void *k, const void *v,
                              const void *o, const void *dout, const float *lse, void *dq, void *dk, void *dv,
                              void *workspace, size_t ws_bytes, void *stream);

/* ---------------------------------------------------------------- instrumentation
 * (no paper counterpart: measurement support for benchmarks and tests)
 * Kernels of this library, as counted and timed below. */
typedef enum {
    BLA_K_TABLES = 0,      /* fp32 interpolation/phase tables (every call) */
    BLA_K_TABLES_BF16,     /* bf16 operand tables of the tensor-core path */
    BLA_K_PREPASS,         /* per-segment state deltas (tcgen05 GEMM) */
    BLA_K_SCAN,            /* states entering each segment */
    BLA_K_KPASS,           /* K pass: scores, softmax, slot probabilities (tcgen05) */
    BLA_K_VPASS,           /* V pass: outputs (tcgen05) */
    BLA_K_FWD_F32,         /* fp32 chunked forward (CUDA cores) */
    BLA_K_DECODE,          /* decode step */
    BLA_K_BWD,             /* backward kernels */
    BLA_K_DECAY,           /* state-decay kernels (table, K scan, lse, V scan, decode) */
    BLA_K_COUNT
} bla_kernel_id;

/* Kernels launched by this library in this process so far. */
long long bla_kernel_launches(void);

/* on != 0: from now on record a CUDA event pair around every kernel launch, on the
 * launch's stream (two event records per launch; off by default). */
bla_status bla_profile_enable(int on);

/* Synchronise the recorded events, add each launch's duration (ms) to ms[kernel] and
 * 1 to launches[kernel] (arrays of BLA_K_COUNT, zeroed by the caller), then forget them. */
bla_status bla_profile_collect(double *ms, int *launches);

/* Synchronise `stream` and report (then clear) the library's device error word:
 * BLA_OK; BLA_ERR_TIMEOUT if a bounded wait gave up since the last call; or
 * BLA_ERR_CUDA if a kernel refused to run because its dynamic shared memory base
 * was not 1024-byte aligned. */
bla_status bla_device_error(void *stream);

/* Self-test of the failure path (no paper counterpart): launch one CTA whose bounded mbarrier
 * wait, on a barrier nothing ever arrives at, gives up after about limit_ms milliseconds (1 to
 * 1000) and records the timeout in the device error word, exactly as a kernel of the library does
 * when a wait runs out.  The next bla_device_error(stream) then returns BLA_ERR_TIMEOUT, and the
 * context stays usable.  Returns BLA_ERR_INVALID for a limit out of range. */
bla_status bla_selftest_wait_timeout(int limit_ms, void *stream);

/* Static description of a status code. */
const char *bla_status_string(bla_status s);

/* Description of the most recent failure on the calling thread ("" if none). */
const char *bla_last_error_string(void);

#ifdef __cplusplus
}
#endif

#endif /* BLA_GB300_H */
