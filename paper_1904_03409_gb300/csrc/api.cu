// api.cu -- the C ABI (include/stacklstm.h): argument checks, workspace ownership and
// the order of launches for forward and backward. All arithmetic runs in the kernels of
// index_kernels.cu, fp32_path.cu and bf16_path.cu.
#include <stdio.h>

#include <algorithm>
#include <new>

#include "common.cuh"

namespace {

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) cudaSetDevice(dev);
    }
    ~DeviceGuard()
    {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

sl_status fail(stacklstm *s, sl_status st, const char *msg)
{
    if (s) s->last_error = msg ? msg : "";
    return st;
}

sl_status cuda_fail(stacklstm *s, cudaError_t e, const char *where)
{
    if (s) {
        char buf[256];
        snprintf(buf, sizeof buf, "%s: %s", where, cudaGetErrorString(e));
        s->last_error = buf;
    }
    return SL_ERR_CUDA;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

size_t elem_size(sl_dtype dt) { return dt == SL_BF16 ? 2 : 4; }

void free_all(stacklstm *s)
{
    for (void *p : s->allocs) cudaFree(p);
    s->allocs.clear();
}

template <typename P>
bool alloc(stacklstm *s, P **out, size_t bytes)
{
    void *p = nullptr;
    if (bytes == 0) bytes = 16;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
        cudaGetLastError();  // clear the sticky-free allocation error
        return false;
    }
    s->allocs.push_back(p);
    *out = (P *)p;
    return true;
}

// Records a CUDA event pair around one phase on the handle's stream when timing is on;
// always adds the phase's kernel launches to its count.
struct Phase {
    stacklstm *s;
    int ph;
    long long l0;
    cudaEvent_t a = nullptr;
    Phase(stacklstm *s_, int ph_) : s(s_), ph(ph_), l0(s_->launches)
    {
        if (s->timing) {
            a = take_event(s);
            if (a) cudaEventRecord(a, s->stream);
        }
    }
    ~Phase()
    {
        s->phase_launches[ph] += s->launches - l0;
        if (a) {
            cudaEvent_t b = take_event(s);
            if (b) {
                cudaEventRecord(b, s->stream);
                s->pending.push_back({ph, a, b});
            } else {
                s->event_pool.push_back(a);
            }
        }
    }
    static cudaEvent_t take_event(stacklstm *s)
    {
        if (!s->event_pool.empty()) {
            cudaEvent_t e = s->event_pool.back();
            s->event_pool.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        return e;
    }
};

// Folds completed event pairs into the per-phase totals (the stream must be idle).
void collect_timing(stacklstm *s)
{
    for (auto &p : s->pending) {
        float ms = 0.0f;
        if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) s->phase_ms[p.phase] += ms;
        s->event_pool.push_back(p.a);
        s->event_pool.push_back(p.b);
    }
    s->pending.clear();
    cudaGetLastError();
}

// Reads back the device error flag (synchronizing the stream) and clears it.
sl_status read_status(stacklstm *s)
{
    int32_t h = 0;
    cudaError_t e = cudaMemcpyAsync(&h, s->err, sizeof h, cudaMemcpyDeviceToHost, s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "synchronize");
    if (h != SL_OK) {
        e = cudaMemsetAsync(s->err, 0, sizeof(int32_t), s->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
        if (e != cudaSuccess) return cuda_fail(s, e, "clear status");
        const char *what = h == SL_ERR_OP ? "op outside {-1, 0, +1}"
                           : h == SL_ERR_UNDERFLOW ? "pop at stack depth 0"
                           : h == SL_ERR_TIMEOUT ? "device-side wait ran out"
                           : "device error";
        return fail(s, (sl_status)h, what);
    }
    return SL_OK;
}

// ---- the phases of a forward and a backward call, shared by the single and grouped calls

// Argument checks, the index prepass and the forward setup (weight packing, initial state).
sl_status fwd_begin(stacklstm *s, const sl_forward_args &a)
{
    s->last_error.clear();
    if (!a.x || !a.ops || !a.h0 || !a.c0 || !a.W || !a.bias || !a.p_final)
        return fail(s, SL_ERR_ARG, "x, ops, h0, c0, W, bias and p_final are required");
    const void *ptrs[] = {a.x, a.h0, a.c0, a.W, a.bias, a.h_stack, a.c_stack, a.p_final, a.p_traj, a.src, a.y};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(s, SL_ERR_ARG, "tensor pointers must be 16-byte aligned");
    cudaError_t e;
    s->fwd_done = 0;
    // the initial state and the weight packing do not depend on the index prepass, so they
    // run on the side stream at the same time (launched after the prepass, whose few blocks
    // then reach the SMs first); the caller's stream waits for them before the forward steps
    if ((e = cudaEventRecord(s->aux_go, s->stream))) return cuda_fail(s, e, "forward setup");
    {
        Phase ph(s, SL_PHASE_PREPASS);
        if ((e = sl::launch_prepass(s, a.ops, a.p_final))) return cuda_fail(s, e, "prepass");
        s->Tr = s->T;
        // push-only mode: each instance's pushes as a virtual timeline
        if (s->push_only && (e = sl::launch_compact(s))) return cuda_fail(s, e, "push-only indices");
    }
    {
        if ((e = cudaStreamWaitEvent(s->side, s->aux_go, 0))) return cuda_fail(s, e, "forward setup");
        const cudaStream_t main = s->stream;
        s->stream = s->side;
        {
            Phase ph(s, SL_PHASE_FWD_SETUP);
            e = s->dt == SL_BF16
                    ? sl::bf16_forward_setup_state(s, (const __nv_bfloat16 *)a.h0, a.c0, (const __nv_bfloat16 *)a.W)
                    : sl::fp32_forward_setup(s, (const float *)a.h0, a.c0, (const float *)a.W);
        }
        s->stream = main;
        if (e) return cuda_fail(s, e, "forward setup");
        if ((e = cudaEventRecord(s->aux_done, s->side))) return cuda_fail(s, e, "forward setup");
    }
    if (s->push_only) {
        // the step count the kernels run is read back here (the one synchronization of this
        // mode's forward)
        Phase ph(s, SL_PHASE_PREPASS);
        if ((e = sl::read_virtual_steps(s))) return cuda_fail(s, e, "push-only indices");
    }
    if (s->dt == SL_BF16) {
        Phase ph(s, SL_PHASE_FWD_SETUP);
        // the x tensor maps (push-only mode: the virtual steps' inputs, gathered after the
        // compaction)
        if ((e = sl::bf16_forward_setup_x(s, (const __nv_bfloat16 *)a.x))) return cuda_fail(s, e, "forward setup");
    }
    if ((e = cudaStreamWaitEvent(s->stream, s->aux_done, 0))) return cuda_fail(s, e, "forward setup");
    return SL_OK;
}

// The gradient history is cleared on the side stream while the forward runs (the forward
// leaves most of the memory bandwidth unused); the side stream first waits for `side_go`,
// recorded on the caller's stream before the forward steps (a previous backward reads it).
sl_status fwd_clear(stacklstm *s)
{
    // the rows the kernels use: T + 1, or in push-only mode the virtual steps' Tr + 1
    const size_t hist_bytes = sizeof(float) * (size_t)(s->Tr + 1) * s->B * s->H;
    cudaError_t e;
    if ((e = cudaStreamWaitEvent(s->side, s->side_go, 0)) ||
        (e = cudaMemsetAsync(s->dhist_h, 0, hist_bytes, s->side)) ||
        (e = cudaMemsetAsync(s->dhist_c, 0, hist_bytes, s->side)) || (e = cudaEventRecord(s->cleared, s->side)))
        return cuda_fail(s, e, "clear");
    s->clear_queued = 1;
    return SL_OK;
}

sl_status fwd_steps(stacklstm *s, const sl_forward_args &a)
{
    Phase ph(s, SL_PHASE_FORWARD);
    cudaError_t e;
    if ((e = cudaEventRecord(s->side_go, s->stream))) return cuda_fail(s, e, "forward");
    if (s->dt == SL_FP32)
        e = sl::fp32_forward_steps(s, (const float *)a.x, (const float *)a.W, a.bias);
    else
        e = sl::bf16_forward_steps(s, a.bias);
    if (e) return cuda_fail(s, e, "forward");
    return fwd_clear(s);
}

// The optional outputs: final pointers, trajectories, provenance, y, the slot-indexed stack.
sl_status fwd_end(stacklstm *s, const sl_forward_args &a)
{
    const int T = s->T, B = s->B, H = s->H;
    const size_t es = elem_size(s->dt);
    cudaError_t e;
    {
        Phase ph(s, SL_PHASE_OUTPUTS);
        if (!s->pfinal_written && (e = cudaMemcpyAsync(a.p_final, s->p_traj + (size_t)T * B, sizeof(int32_t) * B,
                                 cudaMemcpyDeviceToDevice, s->stream)))
            return cuda_fail(s, e, "p_final");
        if (a.p_traj && (e = cudaMemcpyAsync(a.p_traj, s->p_traj, sizeof(int32_t) * (T + 1) * B,
                                             cudaMemcpyDeviceToDevice, s->stream)))
            return cuda_fail(s, e, "p_traj");
        if (a.src && (e = cudaMemcpyAsync(a.src, s->top, sizeof(int32_t) * (T + 1) * B, cudaMemcpyDeviceToDevice,
                                          s->stream)))
            return cuda_fail(s, e, "src");
        // history index of the top after each step and of each slot's last write (in
        // push-only mode: virtual indices, and each slot's last push, as in Sec. 2)
        const int32_t *ytop = s->push_only ? s->vy : s->top, *slots = s->push_only ? s->vslot : s->slot_last;
        if (a.y && (e = sl::launch_gather_rows(s, ytop + B, T * B, es, s->hist_h, a.y, H)))
            return cuda_fail(s, e, "y");
        if (a.h_stack && (e = sl::launch_gather_rows(s, slots, (T + 1) * B, es, s->hist_h, a.h_stack, H)))
            return cuda_fail(s, e, "h_stack");
        if (a.c_stack && (e = sl::launch_gather_rows(s, slots, (T + 1) * B, 4, s->hist_c, a.c_stack, H)))
            return cuda_fail(s, e, "c_stack");
    }
    s->fwd_done = 1;
    return SL_OK;
}

// Argument checks, the cleared and seeded gradient history, the last step's pointwise
// backward (and, push-only mode, the zero dx rows of non-push steps).
sl_status bwd_begin(stacklstm *s, const sl_backward_args &a)
{
    s->last_error.clear();
    if (!s->fwd_done) return fail(s, SL_ERR_STATE, "backward needs a completed forward on this handle");
    const void *ptrs[] = {a.d_top_h, a.dy, a.dx, a.dh0, a.dc0, a.dW, a.dbias};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(s, SL_ERR_ARG, "tensor pointers must be 16-byte aligned");
    // the rows the kernels use: T + 1, or in push-only mode the virtual steps' Tr + 1
    const size_t hist_bytes = sizeof(float) * (size_t)(s->Tr + 1) * s->B * s->H;
    cudaError_t e;
    Phase ph(s, SL_PHASE_BWD_SETUP);
    if (s->clear_queued) {
        // cleared on the side stream during the forward
        if ((e = cudaStreamWaitEvent(s->stream, s->cleared, 0))) return cuda_fail(s, e, "clear");
        s->clear_queued = 0;
    } else {
        if ((e = cudaMemsetAsync(s->dhist_h, 0, hist_bytes, s->stream))) return cuda_fail(s, e, "clear");
        if ((e = cudaMemsetAsync(s->dhist_c, 0, hist_bytes, s->stream))) return cuda_fail(s, e, "clear");
    }
    // bf16 without per-step dy: the final tops' seeds go in with the last step's pointwise
    // backward (the same element owners, one launch fewer)
    const bool seed_in_pointwise = s->dt == SL_BF16 && !a.dy;
    if (!seed_in_pointwise && (e = sl::launch_seed_grads(s, a.d_top_h, a.dy))) return cuda_fail(s, e, "seed");
    if (s->dt == SL_BF16 && (e = sl::bf16_backward_setup(s, seed_in_pointwise ? a.d_top_h : nullptr)))
        return cuda_fail(s, e, "backward setup");
    // push-only mode: the dx rows of steps that do not push are zero; the contraction
    // writes the others. (Zeroing them on the side stream during the step launch slowed
    // the weight gradient that follows by twice the zeroing's own time.)
    if (s->push_only && (e = sl::launch_zero_nonpush_rows(s, a.dx))) return cuda_fail(s, e, "dx rows");
    return SL_OK;
}

sl_status bwd_steps(stacklstm *s, const sl_backward_args &a, bool *dx_done)
{
    Phase ph(s, SL_PHASE_BACKWARD);
    cudaError_t e = s->dt == SL_FP32 ? sl::fp32_backward_steps(s) : sl::bf16_backward_steps(s, a.dx, dx_done);
    return e ? cuda_fail(s, e, "backward") : SL_OK;
}

// dx (unless the step launch computed it on otherwise idle SMs), dW and dbias, dh0 and dc0.
sl_status bwd_end(stacklstm *s, const sl_backward_args &a, bool dx_done)
{
    const int B = s->B, H = s->H;
    cudaError_t e;
    // dx and dW both only read the gate gradients, so dx runs on the side stream at the same
    // time as dW; the caller's stream waits for it
    const bool side_dx = !dx_done && a.dx;
    if (side_dx) {
        if ((e = cudaEventRecord(s->aux_go, s->stream)) || (e = cudaStreamWaitEvent(s->side, s->aux_go, 0)))
            return cuda_fail(s, e, "dx");
        const cudaStream_t main = s->stream;
        s->stream = s->side;
        {
            Phase ph(s, SL_PHASE_DX);
            e = s->dt == SL_FP32 ? sl::fp32_dx(s, a.dx) : sl::bf16_dx(s, a.dx);
        }
        s->stream = main;
        if (e) return cuda_fail(s, e, "dx");
        if ((e = cudaEventRecord(s->aux_done, s->side))) return cuda_fail(s, e, "dx");
    } else if (!dx_done) {
        Phase ph(s, SL_PHASE_DX);
        e = s->dt == SL_FP32 ? sl::fp32_dx(s, a.dx) : sl::bf16_dx(s, a.dx);
        if (e) return cuda_fail(s, e, "dx");
    }
    {
        Phase ph(s, SL_PHASE_DW);
        e = s->dt == SL_FP32 ? sl::fp32_dw(s, a.dW, a.dbias) : sl::bf16_dw(s, a.dW, a.dbias);
        if (e) return cuda_fail(s, e, "dW");
    }
    if (side_dx && (e = cudaStreamWaitEvent(s->stream, s->aux_done, 0))) return cuda_fail(s, e, "dx");
    // slot 0 always holds the initial state, which is history row 0
    if (a.dh0 && (e = cudaMemcpyAsync(a.dh0, s->dhist_h, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return cuda_fail(s, e, "dh0");
    if (a.dc0 && (e = cudaMemcpyAsync(a.dc0, s->dhist_c, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return cuda_fail(s, e, "dc0");
    return SL_OK;
}

// Grouped calls: the members' streams join the first member's stream before the one step
// launch (before = true), and wait for it afterwards.
sl_status join_streams(stacklstm *const *hs, int n, bool before)
{
    cudaError_t e;
    for (int m = 1; m < n; ++m) {
        stacklstm *from = before ? hs[m] : hs[0], *to = before ? hs[0] : hs[m];
        if ((e = cudaEventRecord(from->join, from->stream)) || (e = cudaStreamWaitEvent(to->stream, from->join, 0)))
            return cuda_fail(hs[m], e, "stream join");
    }
    return SL_OK;
}

sl_status check_group(int n, const stacklstm_t *hs, const void *args)
{
    if (n < 1 || n > kMaxGroup || !hs || !args) return SL_ERR_ARG;
    for (int m = 0; m < n; ++m) {
        if (!hs[m]) return SL_ERR_ARG;
        for (int k = 0; k < m; ++k)
            if (hs[k] == hs[m]) return fail(hs[m], SL_ERR_ARG, "a handle appears twice in the group");
        if (hs[m]->device != hs[0]->device) return fail(hs[m], SL_ERR_ARG, "the group's handles share one device");
    }
    return SL_OK;
}

}  // namespace

namespace sl {
cudaError_t configure_prepass(stacklstm *s);
}

extern "C" {

const char *stacklstm_status_string(sl_status st)
{
    switch (st) {
    case SL_OK: return "ok";
    case SL_ERR_ARG: return "invalid argument";
    case SL_ERR_OP: return "op outside {-1, 0, +1}";
    case SL_ERR_UNDERFLOW: return "pop at stack depth 0";
    case SL_ERR_STATE: return "backward without a forward";
    case SL_ERR_CUDA: return "CUDA error";
    case SL_ERR_TIMEOUT: return "device-side wait timed out";
    case SL_ERR_UNSUPPORTED: return "unsupported sizes or device";
    case SL_ERR_OOM: return "out of device memory";
    }
    return "unknown status";
}

const char *stacklstm_last_error(stacklstm_t s) { return s ? s->last_error.c_str() : "null handle"; }

const char *stacklstm_plan(stacklstm_t s) { return s ? s->plan.c_str() : "null handle"; }

sl_status stacklstm_create(stacklstm_t *out, int T, int B, int I, int H, sl_dtype dtype, int device,
                           void *stream)
{
    if (!out) return SL_ERR_ARG;
    *out = nullptr;
    if (T < 1 || B < 1 || I < 1 || H < 1 || (dtype != SL_FP32 && dtype != SL_BF16)) return SL_ERR_ARG;
    // 32-bit launch-shape limits and int32 history indices
    if (B > 65535 || (long long)T * B > (1LL << 31) - 1 || T > (1 << 30)) return SL_ERR_UNSUPPORTED;
    if (dtype == SL_BF16 && sl::bf16_unsupported(T, B, I, H)) return SL_ERR_UNSUPPORTED;

    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
        cudaGetLastError();
        return SL_ERR_ARG;
    }
    DeviceGuard g(device);
    stacklstm *s = new (std::nothrow) stacklstm;
    if (!s) return SL_ERR_OOM;
    s->T = T; s->B = B; s->I = I; s->H = H; s->dt = dtype; s->device = device;
    s->Tr = T;
    s->stream = (cudaStream_t)stream;
    if (cudaDeviceGetAttribute(&s->num_sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) {
        delete s;
        return SL_ERR_UNSUPPORTED;
    }
    const size_t TB = (size_t)T * B, T1B = (size_t)(T + 1) * B, K = (size_t)I + H, G = 4 * (size_t)H;
    const size_t es = elem_size(dtype);
    bool ok = alloc(s, &s->p_traj, T1B * 4) && alloc(s, &s->top, T1B * 4) && alloc(s, &s->slot_last, T1B * 4) &&
              alloc(s, &s->err, 16) && alloc(s, &s->hist_h, T1B * H * es) && alloc(s, &s->hr, dtype == SL_BF16 ? T1B * H * 2 : 16) && alloc(s, &s->hist_c, T1B * H * 4) &&
              alloc(s, &s->gates, dtype == SL_BF16 ? TB * 4 * (((size_t)H + 15) / 16 * 16) * 2 : TB * G * 4) && alloc(s, &s->a_rm, dtype == SL_FP32 ? TB * K * es : 16) &&
              alloc(s, &s->dhist_h, T1B * H * 4) && alloc(s, &s->dhist_c, T1B * H * 4) &&
              alloc(s, &s->dG, TB * G * es);
    if (ok && dtype == SL_FP32) ok = alloc(s, &s->w_fwd, K * G * 4);
    if (ok && dtype == SL_BF16) ok = sl::bf16_prepare(s) == cudaSuccess;
    if (ok) ok = sl::configure_prepass(s) == cudaSuccess;
    if (ok && !s->prepass_smem) ok = alloc(s, &s->slot_scratch, T1B * 4);
    if (ok) ok = cudaMemset(s->err, 0, 16) == cudaSuccess;
    if (ok) ok = cudaStreamCreateWithFlags(&s->side, cudaStreamNonBlocking) == cudaSuccess &&
                 cudaEventCreateWithFlags(&s->side_go, cudaEventDisableTiming) == cudaSuccess &&
                 cudaEventCreateWithFlags(&s->cleared, cudaEventDisableTiming) == cudaSuccess &&
                 cudaEventCreateWithFlags(&s->join, cudaEventDisableTiming) == cudaSuccess &&
                 cudaEventCreateWithFlags(&s->aux_go, cudaEventDisableTiming) == cudaSuccess &&
                 cudaEventCreateWithFlags(&s->aux_done, cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
        if (s->side) cudaStreamDestroy(s->side);
        if (s->side_go) cudaEventDestroy(s->side_go);
        if (s->cleared) cudaEventDestroy(s->cleared);
        if (s->join) cudaEventDestroy(s->join);
        if (s->aux_go) cudaEventDestroy(s->aux_go);
        if (s->aux_done) cudaEventDestroy(s->aux_done);
        cudaGetLastError();
        free_all(s);
        delete s;
        return SL_ERR_OOM;
    }
    s->plan = dtype == SL_BF16 ? sl::bf16_describe(s) : sl::fp32_describe(s);
    *out = s;
    return SL_OK;
}

sl_status stacklstm_set_stream(stacklstm_t s, void *stream)
{
    if (!s) return SL_ERR_ARG;
    s->stream = (cudaStream_t)stream;
    return SL_OK;
}

sl_status stacklstm_set_async(stacklstm_t s, int async)
{
    if (!s) return SL_ERR_ARG;
    s->async = async != 0;
    return SL_OK;
}

sl_status stacklstm_forward(stacklstm_t s, const void *x, const int8_t *ops, const void *h0, const float *c0,
                            const void *W, const float *bias, void *h_stack, float *c_stack, int32_t *p_final,
                            int32_t *p_traj, int32_t *src, void *y)
{
    if (!s) return SL_ERR_ARG;
    DeviceGuard g(s->device);
    const sl_forward_args a{x, ops, h0, c0, W, bias, h_stack, c_stack, p_final, p_traj, src, y};
    sl_status st;
    if ((st = fwd_begin(s, a)) || (st = fwd_steps(s, a)) || (st = fwd_end(s, a))) return st;
    return s->async ? SL_OK : read_status(s);
}

sl_status stacklstm_backward(stacklstm_t s, const float *d_top_h, const float *dy, float *dx, float *dh0,
                             float *dc0, float *dW, float *dbias)
{
    if (!s) return SL_ERR_ARG;
    DeviceGuard g(s->device);
    const sl_backward_args a{d_top_h, dy, dx, dh0, dc0, dW, dbias};
    bool dx_done = false;
    sl_status st;
    if ((st = bwd_begin(s, a)) || (st = bwd_steps(s, a, &dx_done)) || (st = bwd_end(s, a, dx_done))) return st;
    return s->async ? SL_OK : read_status(s);
}

sl_status stacklstm_forward_group(int n, const stacklstm_t *hs, const sl_forward_args *args)
{
    sl_status st = check_group(n, hs, args);
    if (st) return st;
    DeviceGuard g(hs[0]->device);
    stacklstm *h[kMaxGroup];
    for (int m = 0; m < n; ++m) {
        h[m] = hs[m];
        if ((st = fwd_begin(h[m], args[m]))) return st;
    }
    if (n > 1 && sl::bf16_can_group(h, n, true)) {
        const float *bias[kMaxGroup];
        cudaError_t e;
        for (int m = 0; m < n; ++m) {
            bias[m] = args[m].bias;
            if ((e = cudaEventRecord(h[m]->side_go, h[m]->stream))) return cuda_fail(h[m], e, "forward");
        }
        if ((st = join_streams(h, n, true))) return st;
        {
            Phase ph(h[0], SL_PHASE_FORWARD);
            if ((e = sl::bf16_forward_steps_group(h, n, bias, h[0]->stream))) return cuda_fail(h[0], e, "forward");
        }
        if ((st = join_streams(h, n, false))) return st;
        for (int m = 0; m < n; ++m)
            if ((st = fwd_clear(h[m]))) return st;
    } else {
        for (int m = 0; m < n; ++m)
            if ((st = fwd_steps(h[m], args[m]))) return st;
    }
    for (int m = 0; m < n; ++m)
        if ((st = fwd_end(h[m], args[m]))) return st;
    for (int m = 0; m < n; ++m)
        if (!h[m]->async && (st = read_status(h[m]))) return st;
    return SL_OK;
}

sl_status stacklstm_backward_group(int n, const stacklstm_t *hs, const sl_backward_args *args)
{
    sl_status st = check_group(n, hs, args);
    if (st) return st;
    DeviceGuard g(hs[0]->device);
    stacklstm *h[kMaxGroup];
    bool dx_done[kMaxGroup] = {};
    for (int m = 0; m < n; ++m) {
        h[m] = hs[m];
        if ((st = bwd_begin(h[m], args[m]))) return st;
    }
    if (n > 1 && sl::bf16_can_group(h, n, false)) {
        if ((st = join_streams(h, n, true))) return st;
        {
            Phase ph(h[0], SL_PHASE_BACKWARD);
            cudaError_t e = sl::bf16_backward_steps_group(h, n, h[0]->stream);
            if (e) return cuda_fail(h[0], e, "backward");
        }
        if ((st = join_streams(h, n, false))) return st;
    } else {
        for (int m = 0; m < n; ++m)
            if ((st = bwd_steps(h[m], args[m], &dx_done[m]))) return st;
    }
    for (int m = 0; m < n; ++m)
        if ((st = bwd_end(h[m], args[m], dx_done[m]))) return st;
    for (int m = 0; m < n; ++m)
        if (!h[m]->async && (st = read_status(h[m]))) return st;
    return SL_OK;
}

sl_status stacklstm_set_mode(stacklstm_t s, sl_mode mode)
{
    if (!s || (mode != SL_MODE_HOMOGENIZED && mode != SL_MODE_PUSH_ONLY)) return SL_ERR_ARG;
    s->last_error.clear();
    if (mode == SL_MODE_PUSH_ONLY && s->dt != SL_BF16)
        return fail(s, SL_ERR_UNSUPPORTED, "push-only mode runs on the bf16 path");
    DeviceGuard g(s->device);
    cudaError_t e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "synchronize");
    if (mode == SL_MODE_PUSH_ONLY && !s->vtop) {
        const size_t T1B = (size_t)(s->T + 1) * s->B, TB = (size_t)s->T * s->B;
        bool ok = alloc(s, &s->vtop, T1B * 4) && alloc(s, &s->vmap, T1B * 4) && alloc(s, &s->vy, T1B * 4) &&
                  alloc(s, &s->vslot, T1B * 4) && alloc(s, &s->xidx, TB * 4) && alloc(s, &s->vstep, TB * 4) &&
                  alloc(s, &s->x_push, TB * s->I * 2) && alloc(s, &s->kmax, 16);
        if (ok && cudaMallocHost(&s->kmax_host, sizeof(int32_t)) != cudaSuccess) {
            cudaGetLastError();
            s->kmax_host = nullptr;
            ok = false;
        }
        if (!ok) return fail(s, SL_ERR_OOM, "push-only workspace");
    }
    if (mode != (s->push_only ? SL_MODE_PUSH_ONLY : SL_MODE_HOMOGENIZED)) s->fwd_done = 0;
    s->push_only = mode == SL_MODE_PUSH_ONLY;
    const std::string tag = "; push-only steps (dead writes skipped)";
    const size_t at = s->plan.find(tag);
    if (s->push_only && at == std::string::npos) s->plan += tag;
    if (!s->push_only && at != std::string::npos) s->plan.erase(at);
    return SL_OK;
}

sl_status stacklstm_steps_run(stacklstm_t s, int *steps)
{
    if (!s || !steps) return SL_ERR_ARG;
    *steps = s->Tr;
    return SL_OK;
}

sl_status stacklstm_set_timing(stacklstm_t s, int on)
{
    if (!s) return SL_ERR_ARG;
    DeviceGuard g(s->device);
    cudaError_t e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "synchronize");
    collect_timing(s);
    s->timing = on != 0;
    for (int i = 0; i < SL_NUM_PHASES; ++i) {
        s->phase_ms[i] = 0.0;
        s->phase_launches[i] = 0;
    }
    return SL_OK;
}

sl_status stacklstm_get_timing(stacklstm_t s, double *ms, long long *launches, int n)
{
    if (!s || n < 0 || n > SL_NUM_PHASES) return SL_ERR_ARG;
    DeviceGuard g(s->device);
    cudaError_t e = cudaStreamSynchronize(s->stream);
    if (e != cudaSuccess) return cuda_fail(s, e, "synchronize");
    collect_timing(s);
    for (int i = 0; i < n; ++i) {
        if (ms) ms[i] = s->phase_ms[i];
        if (launches) launches[i] = s->phase_launches[i];
    }
    return SL_OK;
}

sl_status stacklstm_status(stacklstm_t s)
{
    if (!s) return SL_ERR_ARG;
    DeviceGuard g(s->device);
    return read_status(s);
}

sl_status stacklstm_destroy(stacklstm_t s)
{
    if (!s) return SL_OK;
    {
        DeviceGuard g(s->device);
        cudaStreamSynchronize(s->stream);
        if (s->side) {
            cudaStreamSynchronize(s->side);
            cudaStreamDestroy(s->side);
        }
        if (s->side_go) cudaEventDestroy(s->side_go);
        if (s->cleared) cudaEventDestroy(s->cleared);
        if (s->join) cudaEventDestroy(s->join);
        if (s->aux_go) cudaEventDestroy(s->aux_go);
        if (s->aux_done) cudaEventDestroy(s->aux_done);
        collect_timing(s);
        for (cudaEvent_t ev : s->event_pool) cudaEventDestroy(ev);
        s->event_pool.clear();
        if (s->kmax_host) cudaFreeHost(s->kmax_host);
        free_all(s);
        cudaGetLastError();
    }
    delete s;
    return SL_OK;
}

}  // extern "C"
