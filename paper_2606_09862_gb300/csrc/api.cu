// api.cu -- the C ABI of libbla_gb300.so: argument checking, workspace layout, dispatch.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "bwd.cuh"
#include "decay.cuh"
#include "fwd_bf16.cuh"
#include "tc.cuh"

namespace bla {

// ------------------------------------------------------------------ launch accounting
namespace {
std::atomic<long long> g_launches{0};
std::atomic<bool> g_prof_on{false};
struct ProfRec {
    int kid;
    cudaEvent_t a, b;
};
std::mutex g_prof_mu;
std::vector<ProfRec> g_prof_recs;       // recorded, not yet collected
std::vector<cudaEvent_t> g_prof_pool;   // idle events

cudaEvent_t pool_get() {
    if (!g_prof_pool.empty()) {
        cudaEvent_t e = g_prof_pool.back();
        g_prof_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}
}  // namespace

ProfScope::ProfScope(int kernel_id, cudaStream_t st) : kid(kernel_id), stream(st), slot(-1) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (!g_prof_on.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    ProfRec r{kernel_id, pool_get(), pool_get()};
    if (!r.a || !r.b) return;
    cudaEventRecord(r.a, st);
    g_prof_recs.push_back(r);
    slot = (int)g_prof_recs.size() - 1;
}

ProfScope::~ProfScope() {
    if (slot < 0) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (slot < (int)g_prof_recs.size()) cudaEventRecord(g_prof_recs[slot].b, stream);
}

NvtxRange::NvtxRange(const char *name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

__device__ int g_dev_error = 0;

// The address is cached per device for the life of the device's primary context (host threads
// may race on the first lookup; both store the same value).
int *device_error_word() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
    static std::atomic<int *> cache[64];
    if (dev < 0 || dev >= 64) return nullptr;
    int *w = cache[dev].load(std::memory_order_acquire);
    if (!w) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_dev_error) != cudaSuccess) return nullptr;
        w = static_cast<int *>(ptr);
        cache[dev].store(w, std::memory_order_release);
    }
    return w;
}

namespace {
thread_local char t_last_error[512] = "";
}  // namespace

void set_last_error(const char *msg) {
    snprintf(t_last_error, sizeof(t_last_error), "%s", msg ? msg : "");
}

namespace {

bla_status fail(bla_status s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
bla_status fail(bla_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
    va_end(ap);
    return s;
}

bla_status cuda_fail(cudaError_t e, const char *what) {
    return fail(BLA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr double kPi = 3.14159265358979323846;
constexpr int kDefaultChunkF32 = 64;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Common parameter checks; fills the derived dimensions.
bla_status check_params(const bla_params *p, OpDims *d) {
    if (!p) return fail(BLA_ERR_INVALID, "params is NULL");
    if (p->B < 1 || p->H < 1) return fail(BLA_ERR_INVALID, "B and H must be >= 1 (got %d, %d)", p->B, p->H);
    if (p->L < 0) return fail(BLA_ERR_INVALID, "L must be >= 0 (got %d)", p->L);
    if (p->d_k < 1 || p->d_v < 1) return fail(BLA_ERR_INVALID, "d_k and d_v must be >= 1");
    if (p->M < 1) return fail(BLA_ERR_INVALID, "M must be >= 1 (got %d)", p->M);
    if (!p->periods && (!(p->window > 0.0) || !isfinite(p->window)))
        return fail(BLA_ERR_INVALID, "window (period T) must be > 0");
    if (!isfinite(p->omega) || !isfinite(p->scale)) return fail(BLA_ERR_INVALID, "omega and scale must be finite");
    if (p->dtype != BLA_F32 && p->dtype != BLA_BF16) return fail(BLA_ERR_INVALID, "dtype must be BLA_F32 or BLA_BF16");
    double Te = fmax(p->window, 2.0 * p->M - 1.0);
    if (p->periods) {
        // one period per head (Alg. 1 and Alg. 3: T in R^H); S must fit under every one of them
        if (p->H > kMaxHeadPeriods)
            return fail(BLA_ERR_UNSUPPORTED, "per-head periods support at most %d heads (H=%d)", kMaxHeadPeriods, p->H);
        double tmin = INFINITY, tmax = 0.0;
        for (int h = 0; h < p->H; ++h) {
            const double T = p->periods[h];
            if (!(T > 0.0) || !isfinite(T)) return fail(BLA_ERR_INVALID, "periods[%d] must be > 0 and finite", h);
            const double Th = fmax(T, 2.0 * p->M - 1.0);
            tmin = fmin(tmin, Th);
            tmax = fmax(tmax, Th);
        }
        if (p->S < 1 || (double)p->S > tmin)
            return fail(BLA_ERR_INVALID, "S must be in [1, min_h T_h] (S=%d, min T_h=%g)", p->S, tmin);
        Te = tmax;
    } else if (p->S < 1 || (double)p->S > Te) {
        return fail(BLA_ERR_INVALID, "S must be in [1, T] (S=%d, T=%g)", p->S, Te);
    }
    if (p->chunk < 0) return fail(BLA_ERR_INVALID, "chunk must be >= 0");
    if (p->phase_mode != BLA_PHASE_LAG && p->phase_mode != BLA_PHASE_ABSOLUTE)
        return fail(BLA_ERR_INVALID, "phase_mode must be BLA_PHASE_LAG or BLA_PHASE_ABSOLUTE (got %d)", p->phase_mode);
    if ((long long)p->B * p->H > (1ll << 31) - 1) return fail(BLA_ERR_INVALID, "B*H too large");
    d->B = p->B; d->H = p->H; d->L = p->L; d->dk = p->d_k; d->dv = p->d_v; d->M = p->M; d->S = p->S;
    d->R2 = 2 * p->M;
    d->T = Te;
    d->w = p->omega > 0.0 ? p->omega : 2.0 * kPi / Te;
    d->scale = (float)(p->scale > 0.0 ? p->scale : 1.0 / sqrt((double)p->d_k));
    d->dtype = p->dtype;
    d->absolute = p->phase_mode == BLA_PHASE_ABSOLUTE;
    d->periods = p->periods;
    d->omega_in = p->omega;
    return BLA_OK;
}


int f32_chunk(const bla_params *p, const OpDims &d) {
    int C = p->chunk > 0 ? p->chunk : kDefaultChunkF32;
    if (d.L > 0 && C > d.L) C = d.L;
    while (C > 1 && forward_f32_smem_bytes(d, C) > 227 * 1024) C /= 2;
    return C < 1 ? 1 : C;
}

bla_status check_ws(void *ws, size_t have, size_t need) {
    if (need == 0) return BLA_OK;
    if (!ws) return fail(BLA_ERR_INVALID, "workspace is NULL but %zu bytes are needed", need);
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(BLA_ERR_INVALID, "workspace must be 256-byte aligned");
    if (have < need) return fail(BLA_ERR_INVALID, "workspace too small: %zu < %zu bytes", have, need);
    return BLA_OK;
}

size_t ws_forward(const bla_params *p, const OpDims &d) {
    if (d.dtype == BLA_F32) {
        int C = f32_chunk(p, d);
        return tables_bytes(d, C) + forward_f32_scratch_bytes(d, C);
    }
    return fwd_bf16_workspace_bytes(d);
}

size_t ws_decode(const OpDims &d) { return tables_bytes(d, 0); }

// One (batch, head) slice at head h's own period (per-head periods, Alg. 1 and Alg. 3: T in R^H), as a
// problem of one head with a shared period.
OpDims one_head(const OpDims &d, int h) {
    HeadPeriods hp;
    head_periods(d, d.omega_in, &hp);
    OpDims o = d;
    o.B = 1;
    o.H = 1;
    o.periods = nullptr;
    if (hp.n > 0) {
        o.T = hp.T[h];
        o.w = hp.w[h];
    }
    return o;
}

// The backward's workspace: with per-head periods the heads run one at a time on one head's workspace.
size_t ws_backward(const OpDims &d) { return bwd_workspace_bytes(d.periods ? one_head(d, 0) : d); }

// Checks shared by the state-decay entry points (Sec. 3.3 on Alg. 1's slot state).
bla_status check_decay(const bla_params *p, OpDims *d, bool forward) {
    bla_status s = check_params(p, d);
    if (s != BLA_OK) return s;
    if (p->phase_mode != BLA_PHASE_ABSOLUTE)
        return fail(BLA_ERR_UNSUPPORTED, "the state decay is defined on the absolute form's slots (Alg. 1): "
                                         "phase_mode must be BLA_PHASE_ABSOLUTE");
    if (d->dk != d->dv || (d->dk != 32 && d->dk != 64 && d->dk != 128))
        return fail(BLA_ERR_UNSUPPORTED, "the decay path needs d_k = d_v in {32, 64, 128} (got %d, %d)", d->dk, d->dv);
    if (d->S > 256) return fail(BLA_ERR_UNSUPPORTED, "the decay path needs S <= 256 (got %d)", d->S);
    if (forward && decay_table_entries(*d) * (d->periods ? (size_t)d->H : 1) > (size_t(1) << 30))
        return fail(BLA_ERR_UNSUPPORTED, "L + T too large for the decay table (L=%d, T=%g)", d->L, d->T);
    // one-dimensional grids: heads x slot blocks (K scan), heads x column blocks (V scan), tokens / 256 (lse)
    const long long bh = (long long)d->B * d->H, imax = (1ll << 31) - 1;
    if (bh * ((d->S + 7) / 8) > imax || bh * (d->dv / 32) > imax || (forward && bh * d->L / 256 + 1 > imax))
        return fail(BLA_ERR_UNSUPPORTED, "B*H too large for the decay kernels' grids (B*H=%lld)", bh);
    return BLA_OK;
}

// bla_selftest_wait_timeout: a bounded wait on a barrier nothing arrives at (kernel id 15 in the
// error word).
__global__ void k_wait_selftest(uint64_t limit_ns, int *err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        tc::mbar_init(&bar, 1);
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !tc::mbar_wait(&bar, 0, limit_ns)) report_device_error(err, DEVERR_MBAR_TIMEOUT | (15 << 4));
}

// ---- host-buffer forward: head groups pipelined over copy streams
constexpr int kHostGroupsMax = 8;
constexpr size_t kHostGroupBytes = 64ull << 20;   // split only when a group still moves >= 64 MB

struct HostPipe {
    cudaStream_t h2d = nullptr, d2h = nullptr;
    cudaEvent_t start = nullptr, in[kHostGroupsMax] = {}, out[kHostGroupsMax] = {}, done = nullptr;
    bool ready = false;
};

// The library's copy streams and events of the current device (created on first use).
cudaError_t host_pipe(HostPipe **pp) {
    static HostPipe pipes[64];
    static std::mutex mu;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(mu);
    HostPipe &h = pipes[dev];
    if (!h.ready) {
        if ((e = cudaStreamCreateWithFlags(&h.h2d, cudaStreamNonBlocking)) != cudaSuccess) return e;
        if ((e = cudaStreamCreateWithFlags(&h.d2h, cudaStreamNonBlocking)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&h.start, cudaEventDisableTiming)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&h.done, cudaEventDisableTiming)) != cudaSuccess) return e;
        for (int i = 0; i < kHostGroupsMax; ++i) {
            if ((e = cudaEventCreateWithFlags(&h.in[i], cudaEventDisableTiming)) != cudaSuccess) return e;
            if ((e = cudaEventCreateWithFlags(&h.out[i], cudaEventDisableTiming)) != cudaSuccess) return e;
        }
        h.ready = true;
    }
    *pp = &h;
    return cudaSuccess;
}

// Head groups of the host-buffer forward: heads [first(g), first(g+1)).
int host_groups(const OpDims &d) {
    const long long BH = (long long)d.B * d.H;
    const size_t elem = d.dtype == BLA_BF16 ? 2 : 4;
    const size_t total = (size_t)BH * d.L * (2 * d.dk + 2 * d.dv) * elem;
    long long n = (long long)(total / kHostGroupBytes);
    if (n > kHostGroupsMax) n = kHostGroupsMax;
    if (n > BH) n = BH;
    return n < 1 ? 1 : (int)n;
}
long long host_group_first(const OpDims &d, int ngroups, int g) { return (long long)d.B * d.H * g / ngroups; }
size_t host_elem(const OpDims &d) { return d.dtype == BLA_BF16 ? 2 : 4; }

// Dimensions of one group's launch: its heads as one batch.
OpDims host_group_dims(const OpDims &d, long long heads) {
    OpDims g = d;
    g.B = 1;
    g.H = (int)heads;
    return g;
}

// Workspace of the host-buffer forward: the largest group's forward workspace, then the device
// copies of q, k, v and o (each 256-aligned).
size_t ws_forward_host_parts(const bla_params *p, const OpDims &d, size_t *fw) {
    const int ng = host_groups(d);
    size_t f = 0;
    for (int g = 0; g < ng; ++g) {
        const long long nh = host_group_first(d, ng, g + 1) - host_group_first(d, ng, g);
        const size_t w = ws_forward(p, host_group_dims(d, nh));
        if (w > f) f = w;
    }
    *fw = align_up(f, 256);
    const size_t BH = (size_t)d.B * d.H, e = host_elem(d);
    return *fw + 2 * align_up(BH * d.L * d.dk * e, 256) + 2 * align_up(BH * d.L * d.dv * e, 256);
}
size_t ws_forward_host(const bla_params *p, const OpDims &d) {
    size_t fw;
    return ws_forward_host_parts(p, d, &fw);
}

// The forward of a validated problem on device buffers (bla_forward_chunked after its checks).
bla_status forward_device(const bla_params *p, const OpDims &d, const void *q, const void *k, const void *v, void *o,
                          float *lse, float *state_out, void *workspace, cudaStream_t st) {
    if (d.dtype == BLA_F32) {
        const int C = f32_chunk(p, d);
        Tables t;
        char *rest = tables_carve(d, C, static_cast<char *>(workspace), &t);
        cudaError_t e = tables_build(d, t, st);
        if (e != cudaSuccess) return cuda_fail(e, "table build");
        e = launch_forward_f32(d, C, t, (const float *)q, (const float *)k, (const float *)v, (float *)o, lse,
                               state_out, reinterpret_cast<float *>(rest), st);
        if (e != cudaSuccess) return cuda_fail(e, "fp32 forward launch");
        return BLA_OK;
    }
    cudaError_t e = fwd_bf16_run(d, q, k, v, o, lse, state_out, workspace, st);
    if (e != cudaSuccess) return cuda_fail(e, "bf16 forward");
    return BLA_OK;
}

}  // namespace

bla_status check_decode(const bla_params *p, long long pos, const void *q, const void *k, const void *v,
                        const float *state, const void *o, OpDims *d) {
    bla_status s = check_params(p, d);
    if (s != BLA_OK) return s;
    if (pos < 0) return fail(BLA_ERR_INVALID, "pos must be >= 0 (got %lld)", pos);
    if (!q || !k || !v || !state || !o) return fail(BLA_ERR_INVALID, "q, k, v, state and o must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(state) || !aligned16(o))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if (d->dk != d->dv || (d->dk != 32 && d->dk != 64 && d->dk != 128))
        return fail(BLA_ERR_UNSUPPORTED, "decode needs d_k = d_v in {32, 64, 128} (got %d, %d)", d->dk, d->dv);
    if (d->S > 256) return fail(BLA_ERR_UNSUPPORTED, "decode needs S <= 256 (got %d)", d->S);
    if (decode_smem_bytes(*d) > 227 * 1024)
        return fail(BLA_ERR_UNSUPPORTED, "decode needs %d bytes of shared memory (M=%d), more than 227 KB",
                    decode_smem_bytes(*d), d->M);
    return BLA_OK;
}

}  // namespace bla

using namespace bla;

extern "C" {

const char *bla_status_string(bla_status s) {
    switch (s) {
    case BLA_OK: return "ok";
    case BLA_ERR_INVALID: return "invalid argument";
    case BLA_ERR_UNSUPPORTED: return "unsupported configuration";
    case BLA_ERR_CUDA: return "CUDA error";
    case BLA_ERR_TIMEOUT: return "device wait timed out";
    default: return "unknown status";
    }
}

const char *bla_last_error_string(void) { return t_last_error; }

size_t bla_workspace_bytes(const bla_params *p, int which) {
    OpDims d;
    if (check_params(p, &d) != BLA_OK) return 0;
    switch (which) {
    case BLA_WS_FORWARD: return ws_forward(p, d);
    case BLA_WS_DECODE: return ws_decode(d);
    case BLA_WS_FORWARD_HOST: return ws_forward_host(p, d);
    case BLA_WS_BACKWARD: return ws_backward(d);
    case BLA_WS_DECAY_FORWARD: return check_decay(p, &d, true) == BLA_OK ? decay_workspace_bytes(d, false) : 0;
    case BLA_WS_DECAY_DECODE: return check_decay(p, &d, false) == BLA_OK ? decay_workspace_bytes(d, true) : 0;
    case BLA_WS_DECAY_BACKWARD: return check_decay(p, &d, true) == BLA_OK ? decay_backward_workspace_bytes(d) : 0;
    default: return 0;
    }
}

bla_status bla_forward_chunked(const bla_params *p, const void *q, const void *k, const void *v, void *o,
                               float *lse, float *state_out, void *workspace, size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_forward_chunked");
    OpDims d;
    bla_status s = check_params(p, &d);
    if (s != BLA_OK) return s;
    if (d.L > 0 && (!q || !k || !v || !o)) return fail(BLA_ERR_INVALID, "q, k, v and o must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse) ||
        !aligned16(state_out))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if (d.dtype == BLA_BF16) {
        const char *why = fwd_bf16_unsupported(d);
        if (why) return fail(BLA_ERR_UNSUPPORTED, "bf16 forward: %s", why);
    }
    if ((s = check_ws(workspace, ws_bytes, ws_forward(p, d))) != BLA_OK) return s;
    return forward_device(p, d, q, k, v, o, lse, state_out, workspace, reinterpret_cast<cudaStream_t>(stream));
}

bla_status bla_forward_chunked_host(const bla_params *p, const void *q, const void *k, const void *v, void *o,
                                    void *workspace, size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_forward_chunked_host");
    OpDims d;
    bla_status s = check_params(p, &d);
    if (s != BLA_OK) return s;
    if (d.L > 0 && (!q || !k || !v || !o)) return fail(BLA_ERR_INVALID, "q, k, v and o must be non-NULL");
    if (d.dtype == BLA_BF16) {
        const char *why = fwd_bf16_unsupported(d);
        if (why) return fail(BLA_ERR_UNSUPPORTED, "bf16 forward: %s", why);
    }
    size_t fw = 0;
    if ((s = check_ws(workspace, ws_bytes, ws_forward_host_parts(p, d, &fw))) != BLA_OK) return s;
    if (d.L == 0) return BLA_OK;
    HostPipe *hp = nullptr;
    cudaError_t e = host_pipe(&hp);
    if (e != cudaSuccess) return cuda_fail(e, "copy streams");
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t BH = (size_t)d.B * d.H, es = host_elem(d);
    const size_t rq = (size_t)d.L * d.dk * es, rv = (size_t)d.L * d.dv * es;   // bytes per head
    char *ws = static_cast<char *>(workspace);
    char *qd = ws + fw, *kd = qd + align_up(BH * rq, 256), *vd = kd + align_up(BH * rq, 256);
    char *od = vd + align_up(BH * rv, 256);
    const char *qh = static_cast<const char *>(q), *kh = static_cast<const char *>(k), *vh = static_cast<const char *>(v);
    char *oh = static_cast<char *>(o);
    // copies start after everything already in `stream` (an earlier call's copies included)
    if ((e = cudaEventRecord(hp->start, st)) != cudaSuccess || (e = cudaStreamWaitEvent(hp->h2d, hp->start, 0)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(hp->d2h, hp->start, 0)) != cudaSuccess)
        return cuda_fail(e, "stream ordering");
    const int ng = host_groups(d);
    for (int g = 0; g < ng; ++g) {
        const long long h0 = host_group_first(d, ng, g), nh = host_group_first(d, ng, g + 1) - h0;
        if ((e = cudaMemcpyAsync(qd + h0 * rq, qh + h0 * rq, nh * rq, cudaMemcpyHostToDevice, hp->h2d)) != cudaSuccess ||
            (e = cudaMemcpyAsync(kd + h0 * rq, kh + h0 * rq, nh * rq, cudaMemcpyHostToDevice, hp->h2d)) != cudaSuccess ||
            (e = cudaMemcpyAsync(vd + h0 * rv, vh + h0 * rv, nh * rv, cudaMemcpyHostToDevice, hp->h2d)) != cudaSuccess ||
            (e = cudaEventRecord(hp->in[g], hp->h2d)) != cudaSuccess || (e = cudaStreamWaitEvent(st, hp->in[g], 0)) != cudaSuccess)
            return cuda_fail(e, "host-to-device copy");
        // the group's heads as one batch; with per-head periods, their periods in the group's order
        // (read on the host only, during the launch)
        OpDims gd = host_group_dims(d, nh);
        std::vector<double> gper;
        if (d.periods) {
            gper.resize((size_t)nh);
            for (long long i = 0; i < nh; ++i) gper[(size_t)i] = d.periods[(h0 + i) % d.H];
            gd.periods = gper.data();
        }
        if ((s = forward_device(p, gd, qd + h0 * rq, kd + h0 * rq, vd + h0 * rv, od + h0 * rv, nullptr, nullptr, ws,
                                st)) != BLA_OK)
            return s;
        if ((e = cudaEventRecord(hp->out[g], st)) != cudaSuccess || (e = cudaStreamWaitEvent(hp->d2h, hp->out[g], 0)) != cudaSuccess ||
            (e = cudaMemcpyAsync(oh + h0 * rv, od + h0 * rv, nh * rv, cudaMemcpyDeviceToHost, hp->d2h)) != cudaSuccess)
            return cuda_fail(e, "device-to-host copy");
    }
    if ((e = cudaEventRecord(hp->done, hp->d2h)) != cudaSuccess || (e = cudaStreamWaitEvent(st, hp->done, 0)) != cudaSuccess)
        return cuda_fail(e, "stream ordering");
    return BLA_OK;
}

bla_status bla_decode_step(const bla_params *p, long long pos, const void *q, const void *k, const void *v,
                           float *state, void *o, void *workspace, size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_decode_step");
    OpDims d;
    bla_status s = check_decode(p, pos, q, k, v, state, o, &d);
    if (s != BLA_OK) return s;
    size_t need = ws_decode(d);
    if ((s = check_ws(workspace, ws_bytes, need)) != BLA_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    Tables t;
    tables_carve(d, 0, static_cast<char *>(workspace), &t);
    cudaError_t e = tables_build(d, t, st);
    if (e != cudaSuccess) return cuda_fail(e, "table build");
    e = launch_decode(d, pos, t, q, k, v, state, o, st);
    if (e != cudaSuccess) return cuda_fail(e, "decode launch");
    return BLA_OK;
}

bla_status bla_decay_forward(const bla_params *p, long long pos0, const void *q, const void *k, const void *v,
                             void *o, float *lse, const float *state_in, float *state_out, void *workspace,
                             size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_decay_forward");
    OpDims d;
    bla_status s = check_decay(p, &d, true);
    if (s != BLA_OK) return s;
    if (pos0 < 0) return fail(BLA_ERR_INVALID, "pos0 must be >= 0 (got %lld)", pos0);
    if (d.L > 0 && (!q || !k || !v || !o)) return fail(BLA_ERR_INVALID, "q, k, v and o must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || (lse && !aligned16(lse)) ||
        (state_in && !aligned16(state_in)) || (state_out && !aligned16(state_out)))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if ((s = check_ws(workspace, ws_bytes, decay_workspace_bytes(d, false))) != BLA_OK) return s;
    cudaError_t e = launch_decay_forward(d, pos0, q, k, v, o, lse, state_in, state_out, workspace,
                                         reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "decay forward launch");
    return BLA_OK;
}

bla_status bla_decay_decode_step(const bla_params *p, long long pos, const void *q, const void *k, const void *v,
                                 float *state, void *o, void *workspace, size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_decay_decode_step");
    OpDims d;
    bla_status s = check_decay(p, &d, false);
    if (s != BLA_OK) return s;
    if (pos < 0) return fail(BLA_ERR_INVALID, "pos must be >= 0 (got %lld)", pos);
    if (!q || !k || !v || !state || !o) return fail(BLA_ERR_INVALID, "q, k, v, state and o must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(state) || !aligned16(o))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if ((s = check_ws(workspace, ws_bytes, decay_workspace_bytes(d, true))) != BLA_OK) return s;
    cudaError_t e = launch_decay_decode(d, pos, q, k, v, state, o, workspace, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "decay decode launch");
    return BLA_OK;
}

bla_status bla_decay_backward(const bla_params *p, long long pos0, const void *q, const void *k, const void *v,
                              const void *o, const void *dout, const float *lse, void *dq, void *dk, void *dv,
                              void *workspace, size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_decay_backward");
    OpDims d;
    bla_status s = check_decay(p, &d, true);
    if (s != BLA_OK) return s;
    if (pos0 < 0) return fail(BLA_ERR_INVALID, "pos0 must be >= 0 (got %lld)", pos0);
    if (d.L > 0 && (!q || !k || !v || !o || !dout || !lse || !dq || !dk || !dv))
        return fail(BLA_ERR_INVALID, "q, k, v, o, dout, lse, dq, dk and dv must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(dout) || !aligned16(lse) ||
        !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    if ((s = check_ws(workspace, ws_bytes, decay_backward_workspace_bytes(d))) != BLA_OK) return s;
    cudaError_t e = launch_decay_backward(d, pos0, q, k, v, o, dout, lse, dq, dk, dv, workspace,
                                          reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "decay backward launch");
    return BLA_OK;
}

bla_status bla_backward(const bla_params *p, const void *q, const void *k, const void *v, const void *o,
                        const void *dout, const float *lse, void *dq, void *dk, void *dv, void *workspace,
                        size_t ws_bytes, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_backward");
    OpDims d;
    bla_status s = check_params(p, &d);
    if (s != BLA_OK) return s;
    if (d.L > 0 && (!q || !k || !v || !o || !dout || !lse || !dq || !dk || !dv))
        return fail(BLA_ERR_INVALID, "q, k, v, o, dout, lse, dq, dk and dv must be non-NULL");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(dout) || !aligned16(lse) ||
        !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
        return fail(BLA_ERR_INVALID, "tensor pointers must be 16-byte aligned");
    const char *why = bwd_unsupported(d.periods ? one_head(d, 0) : d);
    if (why) return fail(BLA_ERR_UNSUPPORTED, "backward: %s", why);
    if ((s = check_ws(workspace, ws_bytes, ws_backward(d))) != BLA_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (!d.periods) {
        cudaError_t e = bwd_run(d, q, k, v, o, dout, lse, dq, dk, dv, workspace, st);
        if (e != cudaSuccess) return cuda_fail(e, "backward");
        return BLA_OK;
    }
    // per-head periods: every (batch, head) slice of the tensors is contiguous; run them one after the
    // other at their own periods on the one-head workspace (stream order keeps the workspace's uses apart)
    const size_t e_sz = d.dtype == BLA_BF16 ? 2 : 4;
    const size_t sq = (size_t)d.L * d.dk * e_sz, sv = (size_t)d.L * d.dv * e_sz;
    for (int b = 0; b < d.B; ++b)
        for (int h = 0; h < d.H; ++h) {
            const size_t i = (size_t)b * d.H + h;
            const OpDims d1 = one_head(d, h);
            cudaError_t e = bwd_run(d1, static_cast<const char *>(q) + i * sq, static_cast<const char *>(k) + i * sq,
                                    static_cast<const char *>(v) + i * sv, static_cast<const char *>(o) + i * sv,
                                    static_cast<const char *>(dout) + i * sv, lse + i * d.L,
                                    static_cast<char *>(dq) + i * sq, static_cast<char *>(dk) + i * sq,
                                    static_cast<char *>(dv) + i * sv, workspace, st);
            if (e != cudaSuccess) return cuda_fail(e, "backward");
        }
    return BLA_OK;
}

bla_status bla_selftest_wait_timeout(int limit_ms, void *stream) {
    t_last_error[0] = 0;
    NvtxRange nvtx("bla_selftest_wait_timeout");
    if (limit_ms < 1 || limit_ms > 1000) return fail(BLA_ERR_INVALID, "limit_ms must be in [1, 1000] (got %d)", limit_ms);
    int *err = device_error_word();
    if (!err) return fail(BLA_ERR_CUDA, "device error word unavailable");
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    {
        ProfScope ps(BLA_K_DECODE, st);   // counted as a launch of the library
        k_wait_selftest<<<1, 32, 0, st>>>((uint64_t)limit_ms * 1000000ull, err);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "self-test launch");
    return BLA_OK;
}

long long bla_kernel_launches(void) { return g_launches.load(); }

bla_status bla_profile_enable(int on) {
    t_last_error[0] = 0;
    g_prof_on.store(on != 0);
    return BLA_OK;
}

bla_status bla_profile_collect(double *ms, int *launches) {
    t_last_error[0] = 0;
    if (!ms || !launches) return fail(BLA_ERR_INVALID, "ms and launches must be non-NULL");
    std::lock_guard<std::mutex> lk(g_prof_mu);
    bla_status st = BLA_OK;
    for (auto &r : g_prof_recs) {
        float t = 0.f;
        cudaError_t e = cudaEventSynchronize(r.b);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
        if (e != cudaSuccess) {
            st = cuda_fail(e, "profile event");
        } else if (r.kid >= 0 && r.kid < BLA_K_COUNT) {
            ms[r.kid] += t;
            launches[r.kid] += 1;
        }
        g_prof_pool.push_back(r.a);
        g_prof_pool.push_back(r.b);
    }
    g_prof_recs.clear();
    return st;
}

bla_status bla_device_error(void *stream) {
    t_last_error[0] = 0;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    int code = 0, zero = 0;
    e = cudaMemcpyFromSymbol(&code, g_dev_error, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "read device error word");
    if (code != 0) {
        e = cudaMemcpyToSymbol(g_dev_error, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "clear device error word");
        if ((code & 15) == DEVERR_SMEM_ALIGN)
            return fail(BLA_ERR_CUDA, "kernel %d found its dynamic shared memory base misaligned (block %d)",
                        (code >> 4) & 15, (code >> 16) & 0xffff);
        return fail(BLA_ERR_TIMEOUT, "device wait gave up (code 0x%x: kind %d, kernel %d, barrier %d, parity %d, block %d)",
                    code, code & 15, (code >> 4) & 15, (code >> 8) & 127, (code >> 15) & 1, (code >> 16) & 0xffff);
    }
    return BLA_OK;
}

}  // extern "C"
