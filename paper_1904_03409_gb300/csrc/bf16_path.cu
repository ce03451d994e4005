// bf16_path.cu -- the homogenized StackLSTM step on sm_103a tensor cores.
//
// Forward, one launch per step t (Algorithm 1, no op-dependent branch). A CTA owns 128
// batch rows and U hidden units with all four of their gates (N = 4U gate columns), so
// the LSTM cell runs in the epilogue straight out of tensor memory:
//   1. gather the contraction operand [x_t ; h_read] (h_read = history row top[t], the
//      state at the stack top) into a 128-byte-swizzled shared-memory ring with 16-byte
//      cp.async copies; the packed weight tile streams through the same ring by bulk copy;
//   2. tcgen05.mma (bf16 in, fp32 accumulate) into tensor memory, issued by one thread;
//   3. epilogue: tcgen05.ld of the 4U pre-activations of each row, bias, sigmoid/tanh,
//      c' = f c_read + i g, h' = o tanh(c'); write history row t + 1 (stack slot p_t + 1),
//      and save the activated gates (fp16) for the backward.
// The x_t part of the contraction does not depend on the previous step: with
// programmatic dependent launch it is loaded and multiplied before the step waits for
// its predecessor.
//
// Backward, one launch per step in reverse time (Sec. 5). A CTA owns 128 rows and U
// hidden units of dh_read = dG_t W_h^T (contraction over the 4H gate columns). Its
// epilogue adds dh_read to the gradient of the state step t read (history row top[t]),
// then runs the pointwise backward of step t - 1 for the same rows and units, which now
// has its complete (dh', dc'): it writes dG_{t-1} (bf16) and adds dc_read. Every
// (row, unit) of the gradient history has one owner, so there are no atomics.
//
// After the loop: dx = dG W_x^T (one K-major contraction over all T*B rows) and
// dW = [x ; h_read]^T dG with dbias as one extra all-ones operand row (an MN-major,
// split-K contraction whose partial sums are reduced in a fixed order).
#include <stdlib.h>

#include <algorithm>

#include "common.cuh"
#include "tc.cuh"

namespace sl {
namespace {

using tc::smem_u32;
using tc::sw128;

constexpr int kThreads = 128;  // four warps: one per 32-lane quadrant of tensor memory
constexpr int kRows = 128;     // MMA M: batch rows (or weight rows) per CTA tile
constexpr int kChunk = 64;     // contraction elements per chunk: one 128-byte swizzled row
constexpr uint32_t kAStage = kRows * 128;
constexpr long long kDrainLimit = 4000000000LL;  // wait for own copies / MMAs before exit

// --------------------------------------------------------------------------- smem
struct Ctl {
    uint32_t a0, b0;  // shared addresses of stage 0 of the A and B rings
    uint64_t *full, *empty, *done;
    uint32_t *tmem_slot;
    volatile int *abort;
};

template <int S, int NB>
struct Layout {
    static constexpr uint32_t kB = (uint32_t)NB * 128;
    static constexpr uint32_t kBars = S * (kAStage + kB);
    static constexpr uint32_t kBytes = kBars + (2 * S + 1) * 8 + 16 + 1024;  // + alignment slack
};

template <int S, int NB>
__device__ __forceinline__ Ctl carve(uint8_t *raw)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    Ctl c;
    c.a0 = smem_u32(base);
    c.b0 = c.a0 + S * kAStage;
    uint8_t *bars = base + Layout<S, NB>::kBars;
    c.full = (uint64_t *)bars;
    c.empty = c.full + S;
    c.done = c.empty + S;
    c.tmem_slot = (uint32_t *)(c.done + 1);
    c.abort = (volatile int *)(c.tmem_slot + 1);
    return c;
}

__device__ __forceinline__ void set_abort(const Ctl &c, int32_t *err)
{
    *c.abort = 1;
    atomicCAS(err, 0, (int)SL_ERR_TIMEOUT);
}

template <int S>
__device__ __forceinline__ void prologue(const Ctl &c, uint32_t ncols)
{
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(&c.full[s], 1);
            tc::mbar_init(&c.empty[s], 1);
        }
        tc::mbar_init(c.done, 1);
        *c.abort = 0;
        tc::fence_mbar_init();
    }
    if (threadIdx.x < 32) tc::tmem_alloc(c.tmem_slot, ncols);
}

__device__ __forceinline__ void finish(const Ctl &c, uint32_t tmem, uint32_t ncols)
{
    tc::tc_fence_before();
    __syncthreads();
    if (threadIdx.x < 32) tc::tmem_dealloc(tmem, ncols);
}

template <int N>
struct TmemCols {
    static constexpr uint32_t value = N <= 32 ? 32 : N <= 64 ? 64 : N <= 128 ? 128 : 256;
};

// ---------------------------------------------------------------------- mainloop
// Streams KC contraction chunks through an S-stage ring and accumulates D = A B^T in
// tensor memory. Every thread issues its share of the A-chunk copies (load_a); the B
// chunk either arrives by one bulk copy from a packed tile (kBulkB) or is loaded by the
// threads too (load_b). Thread 0 issues the MMAs (issue(stage, chunk)) and commits each
// chunk to the stage's `empty` barrier. Before chunk `dep_chunk` is loaded every thread
// waits for the preceding grid (programmatic dependent launch). On return the
// accumulator is complete (or the CTA has aborted; *c.abort is then set and uniform).
template <int S, int NB, bool kBulkB, class LoadA, class LoadB, class Issue>
__device__ __forceinline__ void mainloop(const Ctl &c, int KC, const uint8_t *__restrict__ bpack, int dep_chunk,
                                         long long limit, int32_t *err, LoadA load_a, LoadB load_b, Issue issue)
{
    constexpr uint32_t kB = (uint32_t)NB * 128;
    const int tid = threadIdx.x;
    int n_issued = 0, n_waited = 0;  // bulk B copies (thread 0)
    for (int it = 0; it < KC + S - 1; ++it) {
        if (it < KC) {
            const int s = it % S, use = it / S;
            if (use > 0 && !*c.abort)
                if (!tc::mbar_wait(&c.empty[s], (use - 1) & 1, limit, c.abort)) set_abort(c, err);
            if (it == dep_chunk) tc::grid_dep_wait();
            if (!*c.abort) {
                if (kBulkB) {
                    if (tid == 0) {
                        tc::mbar_arrive_expect_tx(&c.full[s], kB);
                        tc::bulk_g2s(c.b0 + s * kB, bpack + (size_t)it * kB, kB, &c.full[s]);
                        ++n_issued;
                    }
                } else {
                    load_b(it, c.b0 + s * kB);
                }
                load_a(it, c.a0 + s * kAStage);
            }
            tc::cp_async_commit();
        }
        const int j = it - (S - 1);
        if (j >= 0) {
            tc::cp_async_wait_dyn(min(it, KC - 1) - j);
            tc::fence_proxy_async();
            __syncthreads();
            if (tid == 0 && !*c.abort) {
                const int s = j % S;
                bool ok = true;
                if (kBulkB) {
                    ok = j < n_issued && tc::mbar_wait(&c.full[s], (j / S) & 1, limit, c.abort);
                    if (ok) ++n_waited;
                }
                if (ok) {
                    tc::tc_fence_after();
                    issue(s, j);
                    tc::mma_commit(&c.empty[s]);
                } else {
                    set_abort(c, err);
                }
            }
        }
    }
    if (tid == 0) {
        tc::mma_commit(c.done);  // arrives once every MMA issued above has completed
        for (int jj = n_waited; jj < n_issued; ++jj)  // bulk copies still in flight after an abort
            tc::mbar_wait(&c.full[jj % S], (jj / S) & 1, kDrainLimit, nullptr);
    }
    tc::cp_async_wait<0>();
    if (!tc::mbar_wait(c.done, 0, limit, nullptr)) {
        set_abort(c, err);
        tc::mbar_wait(c.done, 0, kDrainLimit, nullptr);
    }
    __syncthreads();
    tc::tc_fence_after();
}

// K-major operands, both 128-byte swizzled rows of 64 bf16: four MMAs of K = 16 per chunk
// step through the swizzle atom by advancing the start address 32 bytes.
template <int N>
__device__ __forceinline__ void issue_kmajor(uint32_t tmem, uint32_t a_stage, uint32_t b_stage, int chunk)
{
    constexpr uint32_t idesc = tc::idesc_bf16(N);
#pragma unroll
    for (int k = 0; k < kChunk / 16; ++k)
        tc::mma_bf16(tmem, tc::smem_desc(a_stage + k * 32, 16, 1024), tc::smem_desc(b_stage + k * 32, 16, 1024),
                     idesc, (chunk | k) != 0);
}

// ----------------------------------------------------------------------- helpers
__device__ __forceinline__ float sigm(float z) { return 1.0f / (1.0f + __expf(-z)); }

__device__ __forceinline__ void ld8f(const float *p, float (&v)[8])
{
    const float4 a = *(const float4 *)p, b = *(const float4 *)(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ void st8f(float *p, const float (&v)[8])
{
    *(float4 *)p = make_float4(v[0], v[1], v[2], v[3]);
    *(float4 *)(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
}
__device__ __forceinline__ uint4 pack8_bf16(const float (&v)[8])
{
    uint4 o;
    __nv_bfloat162 t;
    t = __floats2bfloat162_rn(v[0], v[1]); o.x = *(uint32_t *)&t;
    t = __floats2bfloat162_rn(v[2], v[3]); o.y = *(uint32_t *)&t;
    t = __floats2bfloat162_rn(v[4], v[5]); o.z = *(uint32_t *)&t;
    t = __floats2bfloat162_rn(v[6], v[7]); o.w = *(uint32_t *)&t;
    return o;
}
__device__ __forceinline__ uint4 pack8_f16(const float (&v)[8])
{
    uint4 o;
    __half2 t;
    t = __floats2half2_rn(v[0], v[1]); o.x = *(uint32_t *)&t;
    t = __floats2half2_rn(v[2], v[3]); o.y = *(uint32_t *)&t;
    t = __floats2half2_rn(v[4], v[5]); o.z = *(uint32_t *)&t;
    t = __floats2half2_rn(v[6], v[7]); o.w = *(uint32_t *)&t;
    return o;
}
__device__ __forceinline__ void unpack8_f16(uint4 u, float (&v)[8])
{
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(*(const __half2 *)&w[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// ------------------------------------------------------------------ arguments
struct StepArgs {
    int T, B, I, H;
    const __nv_bfloat16 *x;     // [T][B][I]
    const int32_t *top;         // [T+1][B]
    __nv_bfloat16 *hist_h;      // [T+1][B][H]
    float *hist_c;              // [T+1][B][H]
    __half *gates;              // [T][B][4H]
    const float *bias;          // [4H]
    const uint8_t *wpack;       // packed B-operand tiles of this kernel
    float *dhist_h, *dhist_c;   // [T+1][B][H]
    __nv_bfloat16 *dG;          // [T][B][4H]
    int kc;                     // contraction chunks
    long long limit;
    int32_t *err;
};

// ------------------------------------------------------------------ forward step
template <int U, int S>
__global__ void __launch_bounds__(kThreads, 1) fwd_step_tc(StepArgs a, int t)
{
    constexpr int NB = 4 * U;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_src[kRows];
    const Ctl c = carve<S, NB>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x, row0 = blockIdx.y * kRows;
    const int B = a.B, I = a.I, H = a.H;

    prologue<S>(c, kCols);
    // history row each tile row reads (the prepass finished before the first step)
    for (int r = tid; r < kRows; r += kThreads) s_src[r] = row0 + r < B ? a.top[(size_t)t * B + row0 + r] : 0;
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;

    const __nv_bfloat16 *xt = a.x + (size_t)t * B * I;
    auto load_a = [&](int kc, uint32_t dst) {
        // 128 rows x 8 pieces of 16 bytes; 8 consecutive threads cover one 128-byte row
#pragma unroll 4
        for (int p = tid; p < kRows * 8; p += kThreads) {
            const int r = p >> 3, q = p & 7;
            const int b = row0 + r, k = kc * kChunk + q * 8;
            const void *src = a.x;
            uint32_t bytes = 0;
            if (b < B) {
                if (k < I) {
                    src = xt + (size_t)b * I + k;
                    bytes = 16;
                } else if (k < I + H) {
                    src = a.hist_h + ((size_t)s_src[r] * B + b) * H + (k - I);
                    bytes = 16;
                }
            }
            tc::cp_async16(dst + sw128(r, q), src, bytes);
        }
    };
    auto no_b = [](int, uint32_t) {};
    auto issue = [&](int s, int j) {
        issue_kmajor<NB>(tmem, c.a0 + s * kAStage, c.b0 + s * Layout<S, NB>::kB, j);
    };
    const uint8_t *bpack = a.wpack + (size_t)ct * a.kc * NB * 128;
    // chunks that touch h_read depend on the previous step
    mainloop<S, NB, true>(c, a.kc, bpack, I / kChunk, a.limit, a.err, load_a, no_b, issue);
    tc::grid_dep_launch();

    if (!*c.abort) {
        const int r = tid, b = row0 + r;
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
        const int src = s_src[r];
#pragma unroll 1
        for (int cu = 0; cu < U / 8; ++cu) {
            float z[4][8];
#pragma unroll
            for (int g = 0; g < 4; ++g) tc::tmem_ld8(trow + g * U + cu * 8, z[g]);
            const int u = ct * U + cu * 8;
            if (b < B && u < H) {
                float cr[8], cn[8], hn[8], gv[4][8];
                ld8f(a.hist_c + ((size_t)src * B + b) * H + u, cr);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float ig = sigm(z[0][e] + __ldg(a.bias + u + e));
                    const float fg = sigm(z[1][e] + __ldg(a.bias + H + u + e));
                    const float gg = tanhf(z[2][e] + __ldg(a.bias + 2 * H + u + e));
                    const float og = sigm(z[3][e] + __ldg(a.bias + 3 * H + u + e));
                    cn[e] = fmaf(fg, cr[e], ig * gg);
                    hn[e] = og * tanhf(cn[e]);
                    gv[0][e] = ig; gv[1][e] = fg; gv[2][e] = gg; gv[3][e] = og;
                }
                const size_t w = ((size_t)(t + 1) * B + b) * H + u;
                *(uint4 *)(a.hist_h + w) = pack8_bf16(hn);
                st8f(a.hist_c + w, cn);
                __half *gt = a.gates + ((size_t)t * B + b) * 4 * H + u;
#pragma unroll
                for (int g = 0; g < 4; ++g) *(uint4 *)(gt + (size_t)g * H) = pack8_f16(gv[g]);
            }
        }
    }
    finish(c, tmem, kCols);
}

// ------------------------------------------------------------------ backward pieces
// Pointwise backward of step tp for instance b, hidden units u..u+7 (Sec. 5): reads the
// complete gradient (dh', dc') of the state step tp wrote (history row tp + 1), writes
// the gate pre-activation gradients dG_tp and adds dc_read to the state step tp read.
__device__ __forceinline__ void pointwise8(const StepArgs &a, int tp, int b, int u)
{
    const int B = a.B, H = a.H;
    const size_t wr = ((size_t)(tp + 1) * B + b) * H + u;
    const int s1 = a.top[(size_t)tp * B + b];
    const size_t rd = ((size_t)s1 * B + b) * H + u;
    float dh[8], dcn[8], cn[8], cr[8], ig[8], fg[8], gg[8], og[8];
    ld8f(a.dhist_h + wr, dh);
    ld8f(a.dhist_c + wr, dcn);
    ld8f(a.hist_c + wr, cn);
    ld8f(a.hist_c + rd, cr);
    const __half *gt = a.gates + ((size_t)tp * B + b) * 4 * H + u;
    unpack8_f16(*(const uint4 *)(gt), ig);
    unpack8_f16(*(const uint4 *)(gt + H), fg);
    unpack8_f16(*(const uint4 *)(gt + 2 * (size_t)H), gg);
    unpack8_f16(*(const uint4 *)(gt + 3 * (size_t)H), og);
    float d[4][8], dcr[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float tcn = tanhf(cn[e]);
        const float dc = dcn[e] + dh[e] * og[e] * (1.0f - tcn * tcn);
        d[0][e] = dc * gg[e] * ig[e] * (1.0f - ig[e]);
        d[1][e] = dc * cr[e] * fg[e] * (1.0f - fg[e]);
        d[2][e] = dc * ig[e] * (1.0f - gg[e] * gg[e]);
        d[3][e] = dh[e] * tcn * og[e] * (1.0f - og[e]);
        dcr[e] = dc * fg[e];
    }
    __nv_bfloat16 *dg = a.dG + ((size_t)tp * B + b) * 4 * H + u;
#pragma unroll
    for (int g = 0; g < 4; ++g) *(uint4 *)(dg + (size_t)g * H) = pack8_bf16(d[g]);
    float acc[8];
    ld8f(a.dhist_c + rd, acc);
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] += dcr[e];
    st8f(a.dhist_c + rd, acc);
}

// Pointwise backward of the last step (t = T - 1), before the reverse loop.
__global__ void pointwise_last(StepArgs a)
{
    const int groups = a.H / 8;
    const size_t n = (size_t)a.B * groups;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(e / groups), u = (int)(e - (size_t)b * groups) * 8;
        pointwise8(a, a.T - 1, b, u);
    }
}

template <int U, int S>
__global__ void __launch_bounds__(kThreads, 1) bwd_step_tc(StepArgs a, int t)
{
    constexpr int NB = U;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    extern __shared__ uint8_t smem_raw[];
    __shared__ int s_src[kRows];
    const Ctl c = carve<S, NB>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x, row0 = blockIdx.y * kRows;
    const int B = a.B, H = a.H, G = 4 * H;

    prologue<S>(c, kCols);
    for (int r = tid; r < kRows; r += kThreads) s_src[r] = row0 + r < B ? a.top[(size_t)t * B + row0 + r] : 0;
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;

    const __nv_bfloat16 *dgt = a.dG + (size_t)t * B * G;
    auto load_a = [&](int kc, uint32_t dst) {
#pragma unroll 4
        for (int p = tid; p < kRows * 8; p += kThreads) {
            const int r = p >> 3, q = p & 7;
            const int b = row0 + r, n = kc * kChunk + q * 8;
            const bool ok = b < B && n < G;
            tc::cp_async16(dst + sw128(r, q), ok ? (const void *)(dgt + (size_t)b * G + n) : (const void *)a.dG,
                           ok ? 16u : 0u);
        }
    };
    auto no_b = [](int, uint32_t) {};
    auto issue = [&](int s, int j) {
        issue_kmajor<NB>(tmem, c.a0 + s * kAStage, c.b0 + s * Layout<S, NB>::kB, j);
    };
    const uint8_t *bpack = a.wpack + (size_t)ct * a.kc * NB * 128;
    mainloop<S, NB, true>(c, a.kc, bpack, 0, a.limit, a.err, load_a, no_b, issue);
    tc::grid_dep_launch();

    if (!*c.abort) {
        const int r = tid, b = row0 + r;
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
        const int src = s_src[r];
#pragma unroll 1
        for (int cu = 0; cu < U / 8; ++cu) {
            float acc[8];
            tc::tmem_ld8(trow + cu * 8, acc);
            const int u = ct * U + cu * 8;
            if (b < B && u < H) {
                float *d = a.dhist_h + ((size_t)src * B + b) * H + u;
                float v[8];
                ld8f(d, v);
#pragma unroll
                for (int e = 0; e < 8; ++e) v[e] += acc[e];
                st8f(d, v);
                if (t >= 1) pointwise8(a, t - 1, b, u);
            }
        }
    }
    finish(c, tmem, kCols);
}

// ------------------------------------------------------------- input gradient
struct DxArgs {
    const __nv_bfloat16 *dG;  // [R][4H]
    size_t R;
    int I, H, kc;
    const uint8_t *wpack;
    float *dx;  // [R][I]
    long long limit;
    int32_t *err;
};

template <int N, int S>
__global__ void __launch_bounds__(kThreads, 1) dx_tc(DxArgs a)
{
    constexpr uint32_t kCols = TmemCols<N>::value;
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve<S, N>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x;
    const size_t row0 = (size_t)blockIdx.y * kRows;
    const int G = 4 * a.H;
    prologue<S>(c, kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;
    auto load_a = [&](int kc, uint32_t dst) {
#pragma unroll 4
        for (int p = tid; p < kRows * 8; p += kThreads) {
            const int r = p >> 3, q = p & 7;
            const size_t row = row0 + r;
            const int n = kc * kChunk + q * 8;
            const bool ok = row < a.R && n < G;
            tc::cp_async16(dst + sw128(r, q), ok ? (const void *)(a.dG + row * G + n) : (const void *)a.dG,
                           ok ? 16u : 0u);
        }
    };
    auto no_b = [](int, uint32_t) {};
    auto issue = [&](int s, int j) { issue_kmajor<N>(tmem, c.a0 + s * kAStage, c.b0 + s * Layout<S, N>::kB, j); };
    mainloop<S, N, true>(c, a.kc, a.wpack + (size_t)ct * a.kc * N * 128, -1, a.limit, a.err, load_a, no_b, issue);
    if (!*c.abort) {
        const size_t row = row0 + tid;
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int cu = 0; cu < N / 8; ++cu) {
            float v[8];
            tc::tmem_ld8(trow + cu * 8, v);
            const int col = ct * N + cu * 8;
            if (row < a.R && col < a.I) st8f(a.dx + row * a.I + col, v);
        }
    }
    finish(c, tmem, kCols);
}

// ------------------------------------------------------------- weight gradient
// dW_ext[m][n] = sum_r A[r][m] dG[r][n] over r = t * B + b, where A[r] = [x_t ; h_read ; 1]
// (m = I + H is the all-ones row, which yields dbias). Both operands are read MN-major:
// 64 consecutive r per chunk, 64-wide MN blocks of 128-byte swizzled rows.
struct DwArgs {
    int T, B, I, H;
    const __nv_bfloat16 *x, *hist_h, *dG, *ones;
    const int32_t *top;
    size_t R;
    int n_tiles_n, split;
    float *part;  // [split][mt * 128][nt * 256]
    size_t ld_part, rows_part;
    long long limit;
    int32_t *err;
};

template <int S>
__global__ void __launch_bounds__(kThreads, 1) dw_tc(DwArgs a)
{
    constexpr int NB = 256;
    constexpr uint32_t kCols = 256;
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve<S, NB>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int mt = blockIdx.x / a.n_tiles_n, nt = blockIdx.x % a.n_tiles_n, sp = blockIdx.y;
    const int B = a.B, I = a.I, H = a.H, G = 4 * H;
    const size_t RC = (a.R + kChunk - 1) / kChunk;
    const size_t c_lo = RC * sp / a.split, c_hi = RC * (sp + 1) / a.split;
    const int KC = (int)(c_hi - c_lo);
    prologue<S>(c, kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;

    auto load_a = [&](int kc, uint32_t dst) {  // 64 r-rows x (2 blocks x 8 pieces)
#pragma unroll 4
        for (int p = tid; p < kChunk * 16; p += kThreads) {
            const int rr = p >> 4, blk = (p >> 3) & 1, q = p & 7;
            const size_t r = (c_lo + kc) * kChunk + rr;
            const int m = mt * kRows + blk * 64 + q * 8;
            const void *src = a.ones;
            uint32_t bytes = 0;
            if (r < a.R) {
                if (m < I) {
                    src = a.x + r * I + m;
                    bytes = 16;
                } else if (m < I + H) {
                    const size_t b = r % B;
                    src = a.hist_h + ((size_t)a.top[r] * B + b) * H + (m - I);
                    bytes = 16;
                } else if (m == I + H) {
                    bytes = 16;
                }
            }
            tc::cp_async16(dst + blk * 8192 + sw128(rr, q), src, bytes);
        }
    };
    auto load_b = [&](int kc, uint32_t dst) {  // 64 r-rows x (4 blocks x 8 pieces)
#pragma unroll 4
        for (int p = tid; p < kChunk * 32; p += kThreads) {
            const int rr = p >> 5, blk = (p >> 3) & 3, q = p & 7;
            const size_t r = (c_lo + kc) * kChunk + rr;
            const int n = nt * NB + blk * 64 + q * 8;
            const bool ok = r < a.R && n < G;
            tc::cp_async16(dst + blk * 8192 + sw128(rr, q), ok ? (const void *)(a.dG + r * G + n) : (const void *)a.dG,
                           ok ? 16u : 0u);
        }
    };
    auto issue = [&](int s, int j) {
        constexpr uint32_t idesc = tc::idesc_bf16(NB, 1, 1);
        const uint32_t as = c.a0 + s * kAStage, bs = c.b0 + s * Layout<S, NB>::kB;
#pragma unroll
        for (int k = 0; k < kChunk / 16; ++k)  // 16 r-rows = two 8-row groups = 2048 bytes
            tc::mma_bf16(tmem, tc::smem_desc(as + k * 2048, 8192, 1024), tc::smem_desc(bs + k * 2048, 8192, 1024),
                         idesc, (j | k) != 0);
    };
    if (KC > 0) mainloop<S, NB, false>(c, KC, nullptr, -1, a.limit, a.err, load_a, load_b, issue);
    if (!*c.abort) {
        const size_t m = (size_t)mt * kRows + tid;
        float *dst = a.part + ((size_t)sp * a.rows_part + m) * a.ld_part + (size_t)nt * NB;
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int cu = 0; cu < NB / 16; ++cu) {
            float v[16];
            tc::tmem_ld16(trow + cu * 16, v);
            if (KC == 0)
                for (int e = 0; e < 16; ++e) v[e] = 0.0f;
            *(float4 *)(dst + cu * 16) = make_float4(v[0], v[1], v[2], v[3]);
            *(float4 *)(dst + cu * 16 + 4) = make_float4(v[4], v[5], v[6], v[7]);
            *(float4 *)(dst + cu * 16 + 8) = make_float4(v[8], v[9], v[10], v[11]);
            *(float4 *)(dst + cu * 16 + 12) = make_float4(v[12], v[13], v[14], v[15]);
        }
    }
    finish(c, tmem, kCols);
}

// Fixed-order reduction of the split-K partials into dW and dbias.
__global__ void dw_reduce(int K, int G, int split, const float *__restrict__ part, size_t rows_part, size_t ld,
                          float *__restrict__ dW, float *__restrict__ dbias)
{
    const size_t n = (size_t)(K + 1) * G;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const size_t m = e / G, col = e - m * G;
        float acc = 0.0f;
        for (int s = 0; s < split; ++s) acc += part[((size_t)s * rows_part + m) * ld + col];
        if (m < (size_t)K) {
            if (dW) dW[m * G + col] = acc;
        } else if (dbias) {
            dbias[col] = acc;
        }
    }
}

// ------------------------------------------------------------------ packing
// Forward operand: for column tile ct, rows n = g * U + j hold gate g of hidden unit
// ct * U + j; each row is the matching column of W over the contraction [x ; h] (zero
// padded), in 64-element chunks of 128-byte swizzled rows.
__global__ void pack_fwd(const __nv_bfloat16 *__restrict__ W, int I, int H, int U, int KC, int n_ct,
                         __nv_bfloat16 *__restrict__ out)
{
    const int NB = 4 * U, K = I + H, G = 4 * H;
    const size_t n = (size_t)n_ct * KC * NB * kChunk;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int col = (int)(e % kChunk);
        const size_t rowi = e / kChunk;  // (ct * KC + kc) * NB + row
        const int row = (int)(rowi % NB);
        const size_t tile = rowi / NB;
        const int kc = (int)(tile % KC), ct = (int)(tile / KC);
        const int g = row / U, unit = ct * U + row % U, k = kc * kChunk + col;
        const __nv_bfloat16 v = (unit < H && k < K) ? W[(size_t)k * G + g * H + unit] : __float2bfloat16(0.0f);
        const size_t byte = tile * NB * 128 + sw128(row, col >> 3) + (col & 7) * 2;
        out[byte / 2] = v;
    }
}

// Backward operands: for column tile ct, row m is W row (row0 + ct * NB + m) over the 4H
// gate columns (zero padded): W_h rows (row0 = I, rows < I + H) for dh_read, W_x rows
// (row0 = 0, rows < I) for dx.
__global__ void pack_rows(const __nv_bfloat16 *__restrict__ W, int H, int row0, int nrows, int NB, int KC,
                          int n_ct, __nv_bfloat16 *__restrict__ out)
{
    const int G = 4 * H;
    const size_t n = (size_t)n_ct * KC * NB * kChunk;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int col = (int)(e % kChunk);
        const size_t rowi = e / kChunk;
        const int row = (int)(rowi % NB);
        const size_t tile = rowi / NB;
        const int kc = (int)(tile % KC), ct = (int)(tile / KC);
        const int m = ct * NB + row, k = kc * kChunk + col;
        const __nv_bfloat16 v = (m < nrows && k < G) ? W[(size_t)(row0 + m) * G + k] : __float2bfloat16(0.0f);
        const size_t byte = tile * NB * 128 + sw128(row, col >> 3) + (col & 7) * 2;
        out[byte / 2] = v;
    }
}

// ------------------------------------------------------------------ host side
constexpr int kSf32 = 3, kSf16 = 4, kSf8 = 4;  // forward ring depths by U
constexpr int kSb = 4, kSx = 4, kSw = 4;

template <typename Kern, typename... Args>
cudaError_t launch(Kern kernel, dim3 grid, size_t smem, cudaStream_t st, bool pdl, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = pdl ? at : nullptr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <typename Kern>
cudaError_t allow_smem(Kern k, uint32_t bytes)
{
    return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

int pick_dx_n(int I) { return I <= 32 ? 32 : I <= 64 ? 64 : I <= 128 ? 128 : 256; }

unsigned grid_for(const stacklstm *s, size_t n) { return (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 16)); }

StepArgs step_args(stacklstm *s, const __nv_bfloat16 *x, const float *bias, const void *wpack, int kc)
{
    StepArgs a;
    a.T = s->T; a.B = s->B; a.I = s->I; a.H = s->H;
    a.x = x; a.top = s->top;
    a.hist_h = (__nv_bfloat16 *)s->hist_h; a.hist_c = s->hist_c; a.gates = (__half *)s->gates;
    a.bias = bias; a.wpack = (const uint8_t *)wpack;
    a.dhist_h = s->dhist_h; a.dhist_c = s->dhist_c; a.dG = (__nv_bfloat16 *)s->dG;
    a.kc = kc; a.limit = s->wait_limit; a.err = s->err;
    return a;
}

}  // namespace

const char *bf16_unsupported(int T, int B, int I, int H)
{
    (void)T; (void)B;
    if (I % 8 || H % 8) return "bf16 path needs I and H to be multiples of 8";
    return nullptr;
}

cudaError_t bf16_prepare(stacklstm *s)
{
    const int B = s->B, I = s->I, H = s->H, rt = (int)ceil_div(B, kRows), sms = s->num_sms;
    s->uf = (int)ceil_div(H, 32) * rt >= sms ? 32 : (int)ceil_div(H, 16) * rt >= sms / 2 ? 16 : 8;
    s->ub = (int)ceil_div(H, 32) * rt >= sms ? 32 : 16;
    s->kcf = (int)ceil_div(I + H, kChunk);
    s->kcb = (int)ceil_div(4 * H, kChunk);
    s->nx = pick_dx_n(I);
    s->nxt = (int)ceil_div(I, s->nx);
    s->dw_mt = (int)ceil_div(I + H + 1, kRows);
    s->dw_nt = (int)ceil_div(4 * H, 256);
    const size_t RC = ceil_div((size_t)s->T * B, kChunk);
    s->dw_split = (int)std::max<size_t>(1, std::min<size_t>(sms / std::max(1, s->dw_mt * s->dw_nt), RC / 2));
    const char *lim = getenv("STACKLSTM_WAIT_LIMIT_CYCLES");
    s->wait_limit = lim ? atoll(lim) : 4000000000LL;

    const size_t fwd_bytes = (size_t)ceil_div(H, s->uf) * s->kcf * 4 * s->uf * 128;
    const size_t bwd_bytes = (size_t)ceil_div(H, s->ub) * s->kcb * s->ub * 128;
    const size_t dx_bytes = (size_t)s->nxt * s->kcb * s->nx * 128;
    s->dw_part_elems = (size_t)s->dw_split * s->dw_mt * kRows * s->dw_nt * 256;
    void *p;
    cudaError_t e;
    if ((e = cudaMalloc(&p, fwd_bytes))) return e;
    s->allocs.push_back(p); s->w_fwd = p;
    if ((e = cudaMalloc(&p, bwd_bytes))) return e;
    s->allocs.push_back(p); s->w_bwd = p;
    if ((e = cudaMalloc(&p, dx_bytes))) return e;
    s->allocs.push_back(p); s->w_dx = p;
    if ((e = cudaMalloc(&p, s->dw_part_elems * sizeof(float)))) return e;
    s->allocs.push_back(p); s->dw_part = (float *)p;
    if ((e = cudaMalloc(&p, 16))) return e;
    s->allocs.push_back(p); s->ones = p;
    const uint16_t one[8] = {0x3F80, 0, 0, 0, 0, 0, 0, 0};  // bf16 1.0 followed by zeros
    if ((e = cudaMemcpy(s->ones, one, 16, cudaMemcpyHostToDevice))) return e;

    if ((e = allow_smem(fwd_step_tc<32, kSf32>, Layout<kSf32, 128>::kBytes))) return e;
    if ((e = allow_smem(fwd_step_tc<16, kSf16>, Layout<kSf16, 64>::kBytes))) return e;
    if ((e = allow_smem(fwd_step_tc<8, kSf8>, Layout<kSf8, 32>::kBytes))) return e;
    if ((e = allow_smem(bwd_step_tc<32, kSb>, Layout<kSb, 32>::kBytes))) return e;
    if ((e = allow_smem(bwd_step_tc<16, kSb>, Layout<kSb, 16>::kBytes))) return e;
    if ((e = allow_smem(dx_tc<32, kSx>, Layout<kSx, 32>::kBytes))) return e;
    if ((e = allow_smem(dx_tc<64, kSx>, Layout<kSx, 64>::kBytes))) return e;
    if ((e = allow_smem(dx_tc<128, kSx>, Layout<kSx, 128>::kBytes))) return e;
    if ((e = allow_smem(dx_tc<256, kSx>, Layout<kSx, 256>::kBytes))) return e;
    if ((e = allow_smem(dw_tc<kSw>, Layout<kSw, 256>::kBytes))) return e;
    return cudaSuccess;
}

cudaError_t bf16_forward(stacklstm *s, const __nv_bfloat16 *x, const __nv_bfloat16 *h0, const float *c0,
                         const __nv_bfloat16 *W, const float *bias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H;
    cudaError_t e;
    s->x_saved = x;
    if ((e = cudaMemcpyAsync(s->hist_h, h0, sizeof(__nv_bfloat16) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return e;
    if ((e = cudaMemcpyAsync(s->hist_c, c0, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream))) return e;
    const int nctf = (int)ceil_div(H, s->uf), nctb = (int)ceil_div(H, s->ub);
    pack_fwd<<<grid_for(s, (size_t)nctf * s->kcf * 4 * s->uf * kChunk), 256, 0, s->stream>>>(
        W, I, H, s->uf, s->kcf, nctf, (__nv_bfloat16 *)s->w_fwd);
    pack_rows<<<grid_for(s, (size_t)nctb * s->kcb * s->ub * kChunk), 256, 0, s->stream>>>(
        W, H, I, H, s->ub, s->kcb, nctb, (__nv_bfloat16 *)s->w_bwd);
    pack_rows<<<grid_for(s, (size_t)s->nxt * s->kcb * s->nx * kChunk), 256, 0, s->stream>>>(
        W, H, 0, I, s->nx, s->kcb, s->nxt, (__nv_bfloat16 *)s->w_dx);
    s->launches += 3;
    if ((e = cudaGetLastError())) return e;
    const StepArgs a = step_args(s, x, bias, s->w_fwd, s->kcf);
    const dim3 grid(nctf, ceil_div(B, kRows));
    for (int t = 0; t < T; ++t) {
        const bool pdl = t > 0;
        if (s->uf == 32)
            e = launch(fwd_step_tc<32, kSf32>, grid, Layout<kSf32, 128>::kBytes, s->stream, pdl, a, t);
        else if (s->uf == 16)
            e = launch(fwd_step_tc<16, kSf16>, grid, Layout<kSf16, 64>::kBytes, s->stream, pdl, a, t);
        else
            e = launch(fwd_step_tc<8, kSf8>, grid, Layout<kSf8, 32>::kBytes, s->stream, pdl, a, t);
        if (e) return e;
        s->launches += 1;
    }
    return cudaGetLastError();
}

cudaError_t bf16_backward_steps(stacklstm *s)
{
    const int T = s->T, B = s->B, H = s->H;
    cudaError_t e;
    const StepArgs a = step_args(s, (const __nv_bfloat16 *)s->x_saved, nullptr, s->w_bwd, s->kcb);
    pointwise_last<<<grid_for(s, (size_t)B * (H / 8)), 256, 0, s->stream>>>(a);
    s->launches += 1;
    if ((e = cudaGetLastError())) return e;
    const dim3 grid(ceil_div(H, s->ub), ceil_div(B, kRows));
    for (int t = T - 1; t >= 0; --t) {
        const bool pdl = t < T - 1;
        if (s->ub == 32)
            e = launch(bwd_step_tc<32, kSb>, grid, Layout<kSb, 32>::kBytes, s->stream, pdl, a, t);
        else
            e = launch(bwd_step_tc<16, kSb>, grid, Layout<kSb, 16>::kBytes, s->stream, pdl, a, t);
        if (e) return e;
        s->launches += 1;
    }
    return cudaGetLastError();
}

cudaError_t bf16_dx(stacklstm *s, float *dx)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H;
    const size_t R = (size_t)T * B;
    cudaError_t e;
    if (dx) {
        DxArgs d;
        d.dG = (const __nv_bfloat16 *)s->dG; d.R = R; d.I = I; d.H = H; d.kc = s->kcb;
        d.wpack = (const uint8_t *)s->w_dx; d.dx = dx; d.limit = s->wait_limit; d.err = s->err;
        const dim3 g(s->nxt, ceil_div(R, kRows));
        switch (s->nx) {
        case 32: e = launch(dx_tc<32, kSx>, g, Layout<kSx, 32>::kBytes, s->stream, false, d); break;
        case 64: e = launch(dx_tc<64, kSx>, g, Layout<kSx, 64>::kBytes, s->stream, false, d); break;
        case 128: e = launch(dx_tc<128, kSx>, g, Layout<kSx, 128>::kBytes, s->stream, false, d); break;
        default: e = launch(dx_tc<256, kSx>, g, Layout<kSx, 256>::kBytes, s->stream, false, d); break;
        }
        if (e) return e;
        s->launches += 1;
    }
    return cudaGetLastError();
}

cudaError_t bf16_dw(stacklstm *s, float *dW, float *dbias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H;
    const size_t R = (size_t)T * B;
    cudaError_t e;
    if (dW || dbias) {
        DwArgs w;
        w.T = T; w.B = B; w.I = I; w.H = H;
        w.x = (const __nv_bfloat16 *)s->x_saved; w.hist_h = (const __nv_bfloat16 *)s->hist_h;
        w.dG = (const __nv_bfloat16 *)s->dG; w.ones = (const __nv_bfloat16 *)s->ones; w.top = s->top;
        w.R = R; w.n_tiles_n = s->dw_nt; w.split = s->dw_split; w.part = s->dw_part;
        w.ld_part = (size_t)s->dw_nt * 256; w.rows_part = (size_t)s->dw_mt * kRows;
        w.limit = s->wait_limit; w.err = s->err;
        if ((e = launch(dw_tc<kSw>, dim3(s->dw_mt * s->dw_nt, s->dw_split), Layout<kSw, 256>::kBytes, s->stream,
                        false, w)))
            return e;
        dw_reduce<<<grid_for(s, (size_t)(I + H + 1) * 4 * H), 256, 0, s->stream>>>(
            I + H, 4 * H, s->dw_split, s->dw_part, w.rows_part, w.ld_part, dW, dbias);
        s->launches += 2;
    }
    return cudaGetLastError();
}

}  // namespace sl
