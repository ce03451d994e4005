// bf16_path.cu -- the homogenized StackLSTM step on sm_103a tensor cores.
//
// Forward, one launch per step t (Algorithm 1, no op-dependent branch). A CTA owns 128
// batch rows and U hidden units with all four of their gates (N = 4U gate columns), so
// the LSTM cell runs in the epilogue straight out of tensor memory:
//   1. the contraction operand [x_t ; h_read] streams through a ring of 128-byte-swizzled
//      shared-memory stages: x_t tiles by TMA (rows t*B + b are contiguous), h_read rows
//      (history row top[t][b], the state at each stack top) by 16-byte cp.async, one
//      thread per row; the packed weight tile arrives by bulk copy into the same stage;
//   2. tcgen05.mma (bf16 in, fp32 accumulate) into tensor memory, issued by one thread;
//   3. epilogue: tcgen05.ld of each row's 4U pre-activations, bias, sigmoid/tanh,
//      c' = f c_read + i g, h' = o tanh(c'); write history row t + 1 (stack slot p_t + 1)
//      and the activated gates (fp16) for the backward.
// The x_t chunks do not depend on the previous step: with programmatic dependent launch
// they are loaded and multiplied before the step waits for its predecessor.
//
// Backward, one launch per step in reverse time (Sec. 5). A CTA owns 128 rows and U
// hidden units of dh_read = dG_t W_h^T (contraction over the 4H gate columns, dG_t tiles
// by TMA). Its epilogue adds dh_read to the gradient of the state step t read (history
// row top[t]), then runs the pointwise backward of step t - 1 for the same rows and
// units, which now has its complete (dh', dc'): it writes dG_{t-1} (bf16) and adds
// dc_read. Every (row, unit) of the gradient history has one owner: no atomics.
//
// After the loop: dx = dG W_x^T (one K-major contraction over all T*B rows) and
// dW = [x ; h_read]^T dG with dbias as one extra all-ones operand row (an MN-major,
// split-K contraction whose partial sums are reduced in a fixed order).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <stdio.h>
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
constexpr int kMaxStages = 16;
constexpr long long kDrainLimit = 4000000000LL;  // wait for own copies / MMAs before exit

// --------------------------------------------------------------------------- smem
// Dynamic shared memory: [S A stages][S B stages][full[16] empty[16] done][tmem][abort],
// based at the first 1024-byte boundary (128-byte swizzle atoms are 1024 bytes).
struct Ctl {
    uint32_t a0, b0, b_bytes;  // shared addresses of stage 0 of each ring; B stage size
    uint64_t *full, *empty, *done;
    uint32_t *tmem_slot;
    volatile int *abort;
};

__host__ __device__ constexpr uint32_t smem_bytes(int S, int NB)
{
    return 1024 + (uint32_t)S * (kAStage + (uint32_t)NB * 128) + (2 * kMaxStages + 1) * 8 + 16;
}

__device__ __forceinline__ Ctl carve(uint8_t *raw, int S, int NB)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    Ctl c;
    c.b_bytes = (uint32_t)NB * 128;
    c.a0 = smem_u32(base);
    c.b0 = c.a0 + S * kAStage;
    uint8_t *bars = base + S * (kAStage + c.b_bytes);
    c.full = (uint64_t *)bars;
    c.empty = c.full + kMaxStages;
    c.done = c.empty + kMaxStages;
    c.tmem_slot = (uint32_t *)(c.done + 1);
    c.abort = (volatile int *)(c.tmem_slot + 1);
    return c;
}

__device__ __forceinline__ void set_abort(const Ctl &c, int32_t *err)
{
    *c.abort = 1;
    atomicCAS(err, 0, (int)SL_ERR_TIMEOUT);
}

// Barrier init and tensor-memory allocation; ends with a CTA barrier.
__device__ __forceinline__ uint32_t prologue(const Ctl &c, int S, uint32_t ncols)
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
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    return *c.tmem_slot;
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
// tensor memory. Thread 0 issues, per chunk, the TMA tiles and bulk copies of the stage
// (tma(chunk, stage, full_barrier), which also sets the expected bytes) and the MMAs
// (issue(stage, chunk)), committing each chunk to the stage's `empty` barrier. With
// kGather the other threads also copy their share of the A chunk (gather(chunk, stage))
// by cp.async. Before chunk `dep_chunk` is loaded the loaders wait for the preceding
// grid (programmatic dependent launch); every thread has waited on return. On return the
// accumulator is complete, or the CTA has aborted (*c.abort set, uniform).
template <bool kGather, class Tma, class Gather, class Issue>
__device__ __forceinline__ void mainloop(const Ctl &c, int S, int KC, int dep_chunk, long long limit, int32_t *err,
                                         Tma tma, Gather gather, Issue issue)
{
    // Every blocking wait below runs warp-uniformly: a try_wait suspends its whole warp,
    // so a lone issuing lane must never share its warp with spinning lanes.
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int n_issued = 0, n_waited = 0;  // warp 0: chunks whose copies were issued / awaited
    if (kGather || warp == 0) {
        for (int it = 0; it < KC + S - 1; ++it) {
            if (it < KC) {
                const int s = it % S, use = it / S;
                if (use > 0 && !*c.abort)
                    if (!tc::mbar_wait(&c.empty[s], (use - 1) & 1, limit, c.abort)) set_abort(c, err);
                if (it == dep_chunk) tc::grid_dep_wait();
                if (!*c.abort) {
                    if (tid == 0) tma(it, s, &c.full[s]);
                    if (warp == 0) ++n_issued;
                    if (kGather) gather(it, s);
                }
                if (kGather) tc::cp_async_commit();
            }
            const int j = it - (S - 1);
            if (j >= 0) {
                if (kGather) {
                    tc::cp_async_wait_dyn(min(it, KC - 1) - j);
                    tc::fence_proxy_async();
                    __syncthreads();
                }
                if (warp == 0 && !*c.abort) {
                    const int s = j % S;
                    if (j < n_issued && tc::mbar_wait(&c.full[s], (j / S) & 1, limit, c.abort)) {
                        ++n_waited;
                        if (lane == 0) {
                            tc::tc_fence_after();
                            issue(s, j);
                            tc::mma_commit(&c.empty[s]);
                        }
                        __syncwarp();
                    } else {
                        set_abort(c, err);
                    }
                }
            }
        }
    }
    tc::grid_dep_wait();  // every thread: later reads may touch the preceding grid's output
    if (warp == 0) {
        if (lane == 0) tc::mma_commit(c.done);  // arrives once every MMA issued above has completed
        for (int jj = n_waited; jj < n_issued; ++jj)  // copies still in flight after an abort
            tc::mbar_wait(&c.full[jj % S], (jj / S) & 1, kDrainLimit, nullptr);
    }
    if (kGather) tc::cp_async_wait<0>();
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
// Cell nonlinearities of the bf16 path: the hardware tanh approximation (PTX
// tanh.approx.f32, relative error about 2^-11, below the bf16 rounding of h), and the
// logistic sigmoid through the identity sigmoid(z) = 1/2 + tanh(z / 2) / 2.
__device__ __forceinline__ float tanh_hw(float x)
{
    float y;
    asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float sigm(float z) { return fmaf(0.5f, tanh_hw(0.5f * z), 0.5f); }

// L2-coherent read (bypasses L1) of state another CTA or an earlier launch wrote.
__device__ __forceinline__ void ld8f_cg(const float *p, float (&v)[8])
{
    const float4 a = __ldcg((const float4 *)p), b = __ldcg((const float4 *)(p + 4));
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
    int kcx, KC, S;             // x-part chunks, all chunks, ring depth
    const int32_t *top;         // [T+1][B]
    __nv_bfloat16 *hist_h;      // [T+1][B][H]
    __nv_bfloat16 *hr;          // [T+1][B][H] h operand of each step
    float *hist_c;              // [T+1][B][H]
    __half *gates;              // [T][B][4H]
    const float *bias;          // [4H]
    const uint8_t *wpack;       // packed B-operand tiles of this kernel
    float *dhist_h, *dhist_c;   // [T+1][B][H]
    __nv_bfloat16 *dG;          // [T][B][4H]
    long long limit;
    int32_t *err;
};


// Forward epilogue for one tile row and 8 hidden units: the cell on pre-activations z
// (gate blocks i, f, g, o), writes history row t + 1 (h', c'), the gates, and the h
// operand of step t + 1: h' when step t pushed (the new state is the next top), else the
// older top, a row this tile already wrote (hcopy).
__device__ __forceinline__ void fwd_cell8(const StepArgs &a, int t, int b, int u, const float (&z)[4][8],
                                          const float *bias_i, const float *bias_f, const float *bias_g,
                                          const float *bias_o, const float *cr, bool next_is_new, uint4 hcopy)
{
    const int B = a.B, H = a.H;
    float cn[8], hn[8], gv[4][8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float ig = sigm(z[0][e] + bias_i[e]);
        const float fg = sigm(z[1][e] + bias_f[e]);
        const float gg = tanh_hw(z[2][e] + bias_g[e]);
        const float og = sigm(z[3][e] + bias_o[e]);
        cn[e] = fmaf(fg, cr[e], ig * gg);
        hn[e] = og * tanh_hw(cn[e]);
        gv[0][e] = ig; gv[1][e] = fg; gv[2][e] = gg; gv[3][e] = og;
    }
    const size_t w = ((size_t)(t + 1) * B + b) * H + u;
    const uint4 hb = pack8_bf16(hn);
    *(uint4 *)(a.hist_h + w) = hb;
    *(uint4 *)(a.hr + w) = next_is_new ? hb : hcopy;
    st8f(a.hist_c + w, cn);
    __half *gt = a.gates + ((size_t)t * B + b) * 4 * H + u;
#pragma unroll
    for (int g = 0; g < 4; ++g) *(uint4 *)(gt + (size_t)g * H) = pack8_f16(gv[g]);
}

// ------------------------------------------------------------------ forward step
// The contraction runs over [x_t padded to 64 ; h_read padded to 64]: chunks < kcx are
// TMA tiles of x_t, the rest TMA tiles of hr[t] (the h operand the previous step wrote).
template <int U>
__global__ void __launch_bounds__(kThreads, 1)
fwd_step_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_h, StepArgs a, int t)
{
    constexpr int NB = 4 * U;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve(smem_raw, a.S, NB);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x, row0 = blockIdx.y * kRows;
    const int B = a.B, H = a.H, kcx = a.kcx;
    const int b = row0 + tid;
    const bool row_ok = b < B;
    // the prepass ran before the first step: its indices are safe to read early
    const int src = row_ok ? a.top[(size_t)t * B + b] : 0;
    const int s_next = row_ok ? a.top[(size_t)(t + 1) * B + b] : 0;
    const uint32_t tmem = prologue(c, a.S, kCols);

    const uint8_t *bpack = a.wpack + (size_t)ct * a.KC * c.b_bytes;
    auto tma = [&](int it, int s, uint64_t *bar) {
        tc::mbar_arrive_expect_tx(bar, c.b_bytes + kAStage);
        if (it < kcx)
            tc::tma_load_2d(c.a0 + s * kAStage, &tm_x, it * kChunk, t * B + row0, bar);
        else
            tc::tma_load_2d(c.a0 + s * kAStage, &tm_h, (it - kcx) * kChunk, t * B + row0, bar);
        tc::bulk_g2s(c.b0 + s * c.b_bytes, bpack + (size_t)it * c.b_bytes, c.b_bytes, bar);
    };
    auto no_gather = [](int, int) {};
    auto issue = [&](int s, int j) { issue_kmajor<NB>(tmem, c.a0 + s * kAStage, c.b0 + s * c.b_bytes, j); };
    // chunks of hr[t] depend on the previous step
    mainloop<false>(c, a.S, a.KC, kcx, a.limit, a.err, tma, no_gather, issue);
    tc::grid_dep_launch();

    if (!*c.abort) {
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int cu = 0; cu < U / 8; ++cu) {
            float z[4][8];
#pragma unroll
            for (int g = 0; g < 4; ++g) tc::tmem_ld8(trow + g * U + cu * 8, z[g]);
            const int u = ct * U + cu * 8;
            if (row_ok && u < H) {
                float cr[8];
                ld8f_cg(a.hist_c + ((size_t)src * B + b) * H + u, cr);
                const bool is_new = s_next == t + 1;
                const uint4 hc = is_new ? make_uint4(0, 0, 0, 0)
                                        : __ldcg((const uint4 *)(a.hr + ((size_t)s_next * B + b) * H + u));
                float bi[8], bf[8], bg[8], bo[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    bi[e] = __ldg(a.bias + u + e);
                    bf[e] = __ldg(a.bias + H + u + e);
                    bg[e] = __ldg(a.bias + 2 * H + u + e);
                    bo[e] = __ldg(a.bias + 3 * H + u + e);
                }
                fwd_cell8(a, t, b, u, z, bi, bf, bg, bo, cr, is_new, hc);
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
    ld8f_cg(a.dhist_h + wr, dh);
    ld8f_cg(a.dhist_c + wr, dcn);
    ld8f_cg(a.hist_c + wr, cn);
    ld8f_cg(a.hist_c + rd, cr);
    const __half *gt = a.gates + ((size_t)tp * B + b) * 4 * H + u;
    unpack8_f16(*(const uint4 *)(gt), ig);
    unpack8_f16(*(const uint4 *)(gt + H), fg);
    unpack8_f16(*(const uint4 *)(gt + 2 * (size_t)H), gg);
    unpack8_f16(*(const uint4 *)(gt + 3 * (size_t)H), og);
    float d[4][8], dcr[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float tcn = tanh_hw(cn[e]);
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
    ld8f_cg(a.dhist_c + rd, acc);
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

template <int U>
__global__ void __launch_bounds__(kThreads, 1)
bwd_step_tc(const __grid_constant__ CUtensorMap tm_g, StepArgs a, int t)
{
    constexpr int NB = U;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve(smem_raw, a.S, NB);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x, row0 = blockIdx.y * kRows;
    const int B = a.B, H = a.H;
    const int b = row0 + tid;
    const bool row_ok = b < B;
    const int src = row_ok ? a.top[(size_t)t * B + b] : 0;
    const uint32_t tmem = prologue(c, a.S, kCols);

    const uint8_t *bpack = a.wpack + (size_t)ct * a.KC * c.b_bytes;
    auto tma = [&](int it, int s, uint64_t *bar) {
        tc::mbar_arrive_expect_tx(bar, kAStage + c.b_bytes);
        tc::tma_load_2d(c.a0 + s * kAStage, &tm_g, it * kChunk, t * B + row0, bar);
        tc::bulk_g2s(c.b0 + s * c.b_bytes, bpack + (size_t)it * c.b_bytes, c.b_bytes, bar);
    };
    auto no_gather = [](int, int) {};
    auto issue = [&](int s, int j) { issue_kmajor<NB>(tmem, c.a0 + s * kAStage, c.b0 + s * c.b_bytes, j); };
    mainloop<false>(c, a.S, a.KC, 0, a.limit, a.err, tma, no_gather, issue);
    tc::grid_dep_launch();

    if (!*c.abort) {
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int cu = 0; cu < U / 8; ++cu) {
            float acc[8];
            tc::tmem_ld8(trow + cu * 8, acc);
            const int u = ct * U + cu * 8;
            if (row_ok && u < H) {
                float *d = a.dhist_h + ((size_t)src * B + b) * H + u;
                float v[8];
                ld8f_cg(d, v);
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
    size_t R;
    int I, KC, S;
    const uint8_t *wpack;
    float *dx;  // [R][I]
    long long limit;
    int32_t *err;
};

template <int N>
__global__ void __launch_bounds__(kThreads, 1) dx_tc(const __grid_constant__ CUtensorMap tm_g, DxArgs a)
{
    constexpr uint32_t kCols = TmemCols<N>::value;
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve(smem_raw, a.S, N);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int ct = blockIdx.x;
    const size_t row0 = (size_t)blockIdx.y * kRows;
    const uint32_t tmem = prologue(c, a.S, kCols);
    const uint8_t *bpack = a.wpack + (size_t)ct * a.KC * c.b_bytes;
    auto tma = [&](int it, int s, uint64_t *bar) {
        tc::mbar_arrive_expect_tx(bar, kAStage + c.b_bytes);
        tc::tma_load_2d(c.a0 + s * kAStage, &tm_g, it * kChunk, (int)row0, bar);
        tc::bulk_g2s(c.b0 + s * c.b_bytes, bpack + (size_t)it * c.b_bytes, c.b_bytes, bar);
    };
    auto no_gather = [](int, int) {};
    auto issue = [&](int s, int j) { issue_kmajor<N>(tmem, c.a0 + s * kAStage, c.b0 + s * c.b_bytes, j); };
    mainloop<false>(c, a.S, a.KC, -1, a.limit, a.err, tma, no_gather, issue);
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
// 64 consecutive r per chunk; each 64-wide MN block is 64 rows of 128 swizzled bytes.
// dG blocks, x blocks and h blocks (each fully inside x or inside h; the h operand of
// step t is hr[t], rows t * B + b) arrive by TMA; a block straddling x and h, or holding
// the ones row, is copied piece by piece.
struct DwArgs {
    int B, I, H;
    const __nv_bfloat16 *x, *hr, *ones;
    int R;
    int n_tiles_n, split, S;
    float *part;  // [split][mt * 128][nt * 256]
    size_t ld_part, rows_part;
    long long limit;
    int32_t *err;
};

__global__ void __launch_bounds__(kThreads, 1)
dw_tc(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_h,
      const __grid_constant__ CUtensorMap tm_g, DwArgs a)
{
    constexpr int NB = 256;
    constexpr uint32_t kCols = 256;
    constexpr uint32_t kBlk = 64 * 128;  // one MN block of a chunk
    extern __shared__ uint8_t smem_raw[];
    const Ctl c = carve(smem_raw, a.S, NB);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int mt = blockIdx.x / a.n_tiles_n, nt = blockIdx.x % a.n_tiles_n, sp = blockIdx.y;
    const int I = a.I, H = a.H;
    const int RC = (a.R + kChunk - 1) / kChunk;
    const int c_lo = (int)((long long)RC * sp / a.split), c_hi = (int)((long long)RC * (sp + 1) / a.split);
    const int KC = c_hi - c_lo;
    const uint32_t tmem = prologue(c, a.S, kCols);

    auto in_x = [&](int m0) { return m0 + 64 <= I; };
    auto in_h = [&](int m0) { return m0 >= I && m0 + 64 <= I + H; };
    auto tma = [&](int it, int s, uint64_t *bar) {
        const int r0 = (c_lo + it) * kChunk;
        uint32_t bytes = 4 * kBlk;
        for (int blk = 0; blk < 2; ++blk) {
            const int m0 = mt * kRows + blk * 64;
            if (in_x(m0) || in_h(m0)) bytes += kBlk;
        }
        tc::mbar_arrive_expect_tx(bar, bytes);
        for (int blk = 0; blk < 2; ++blk) {
            const int m0 = mt * kRows + blk * 64;
            if (in_x(m0)) tc::tma_load_2d(c.a0 + s * kAStage + blk * kBlk, &tm_x, m0, r0, bar);
            else if (in_h(m0)) tc::tma_load_2d(c.a0 + s * kAStage + blk * kBlk, &tm_h, m0 - I, r0, bar);
        }
        for (int nb = 0; nb < 4; ++nb)
            tc::tma_load_2d(c.b0 + s * c.b_bytes + nb * kBlk, &tm_g, nt * NB + nb * 64, r0, bar);
    };
    // thread -> (r-row rr, block blk): one 128-byte row segment of eight 16-byte pieces
    auto gather = [&](int it, int s) {
        const int rr = tid & 63, blk = tid >> 6;
        const int m0 = mt * kRows + blk * 64;
        if (in_x(m0) || in_h(m0)) return;  // arrives by TMA
        const int r = (c_lo + it) * kChunk + rr;
        const uint32_t dst = c.a0 + s * kAStage + blk * kBlk;
        const bool r_ok = r < a.R;
        const __nv_bfloat16 *hrow = a.hr + (size_t)(r_ok ? r : 0) * H;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int m = m0 + q * 8;
            const void *p = a.ones;
            uint32_t bytes = 0;
            if (r_ok) {
                if (m < I) {
                    p = a.x + (size_t)r * I + m;
                    bytes = 16;
                } else if (m < I + H) {
                    p = hrow + (m - I);
                    bytes = 16;
                } else if (m == I + H) {
                    bytes = 16;
                }
            }
            tc::cp_async16(dst + sw128(rr, q), p, bytes);
        }
    };
    auto issue = [&](int s, int j) {
        constexpr uint32_t idesc = tc::idesc_bf16(NB, 1, 1);
        const uint32_t as = c.a0 + s * kAStage, bs = c.b0 + s * c.b_bytes;
#pragma unroll
        for (int k = 0; k < kChunk / 16; ++k)  // 16 r-rows = two 8-row groups = 2048 bytes
            tc::mma_bf16(tmem, tc::smem_desc(as + k * 2048, kBlk, 1024), tc::smem_desc(bs + k * 2048, kBlk, 1024),
                         idesc, (j | k) != 0);
    };
    if (KC > 0) mainloop<true>(c, a.S, KC, -1, a.limit, a.err, tma, gather, issue);
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


// ------------------------------------------------------------ persistent steps
// One cooperative launch runs all T steps. Each CTA keeps one column tile (U hidden
// units; its weight tile stays in shared memory when it fits) and a fixed set of row
// tiles (rt = slot, slot + n_slot, ...), so every (instance, unit) has one owner for the
// whole launch. The only inter-CTA dependency is within a row tile: step t reads the
// hidden states (forward) or gate gradients (backward) that all column tiles of the row
// tile wrote at the previous step, so each row tile has a counter of completed steps,
// raised with release semantics after a tile's stores and waited on with acquire
// semantics (a bounded spin) before the dependent chunks are loaded.
//
// With cl > 1, the cl CTAs of a thread-block cluster share their row tiles and hold cl
// consecutive column tiles, so they need the same A operand: chunk it is loaded once, by
// cluster rank it % cl, and multicast into the same ring stage of every CTA of the
// cluster. Each CTA arms its own `full` barrier with the chunk's bytes; `empty` counts cl
// arrivals because every CTA commits its MMA completions to the `empty` barrier of all
// CTAs of the cluster, so a stage is refilled only after every consumer drained it.
struct PersistArgs {
    StepArgs s;
    int n_ct, n_rt, n_slot;  // column tiles (a multiple of cl); row tiles; CTAs per column tile
    int w_res;               // 1: weight tile resident in shared memory
    int cl;                  // cluster size along the column tiles (1: no multicast)
    int32_t *cnt;            // [n_rt] completed steps per row tile, zero at launch
};

__host__ __device__ constexpr uint32_t psmem_bytes(int S, int NB, int KC, int w_res)
{
    return 1024 + (w_res ? (uint32_t)KC * NB * 128 : 0u) + (uint32_t)S * kAStage +
           (w_res ? 0u : (uint32_t)S * NB * 128) + (2 * kMaxStages + 2) * 8 + 16;
}

struct PCtl {
    Ctl c;
    uint32_t w0;     // resident weight tile (w_res)
    uint64_t *wbar;  // its bulk-copy barrier
};

__device__ __forceinline__ PCtl pcarve(uint8_t *raw, int S, int NB, int KC, int w_res)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    PCtl p;
    Ctl &c = p.c;
    c.b_bytes = (uint32_t)NB * 128;
    const uint32_t wbytes = w_res ? (uint32_t)KC * c.b_bytes : 0u;
    p.w0 = smem_u32(base);
    c.a0 = p.w0 + wbytes;
    c.b0 = c.a0 + S * kAStage;
    uint8_t *bars = base + wbytes + S * kAStage + (w_res ? 0u : S * c.b_bytes);
    c.full = (uint64_t *)bars;
    c.empty = c.full + kMaxStages;
    c.done = c.empty + kMaxStages;
    p.wbar = c.done + 1;
    c.tmem_slot = (uint32_t *)(p.wbar + 1);
    c.abort = (volatile int *)(c.tmem_slot + 1);
    return p;
}

// Barrier init (empty counts one arrival per CTA of the cluster), tensor-memory
// allocation, then a cluster barrier so no multicast reaches an uninitialised barrier.
__device__ __forceinline__ uint32_t pprologue(const PCtl &pc, int S, uint32_t ncols, int cl)
{
    const Ctl &c = pc.c;
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(&c.full[s], 1);
            tc::mbar_init(&c.empty[s], (uint32_t)cl);
        }
        tc::mbar_init(c.done, 1);
        tc::mbar_init(pc.wbar, 1);
        *c.abort = 0;
        tc::fence_mbar_init();
    }
    if (threadIdx.x < 32) tc::tmem_alloc(c.tmem_slot, ncols);
    tc::tc_fence_before();
    __syncthreads();
    if (cl > 1) tc::cluster_sync();
    tc::tc_fence_after();
    return *c.tmem_slot;
}

// One MMA chunk's completion goes to the stage's empty barrier of every CTA of the cluster.
__device__ __forceinline__ void commit_empty(uint64_t *bar, int cl)
{
    if (cl > 1)
        tc::mma_commit_mc(bar, (uint16_t)((1u << cl) - 1));
    else
        tc::mma_commit(bar);
}

// Loads chunk `it` of a tile into ring slot g: arms this CTA's full barrier with `bytes`
// (A chunk plus this CTA's streamed weight chunk), and, if this CTA is the chunk's issuer,
// loads the A box into every CTA of the cluster. Called by lane 0 of warp 0.
__device__ __forceinline__ void load_a_chunk(const Ctl &c, int s, uint32_t bytes, const CUtensorMap *tm, int c0,
                                             int c1, int it, int cl, uint32_t rank)
{
    tc::mbar_arrive_expect_tx(&c.full[s], bytes);
    if (cl == 1)
        tc::tma_load_2d(c.a0 + s * kAStage, tm, c0, c1, &c.full[s]);
    else if ((uint32_t)(it % cl) == rank)
        tc::tma_load_2d_mc(c.a0 + s * kAStage, tm, c0, c1, &c.full[s], (uint16_t)((1u << cl) - 1));
}

// Bounded spin until *cnt >= target (acquire). False on timeout or abort.
__device__ __forceinline__ bool spin_until(const int32_t *cnt, int target, long long limit, volatile int *abort)
{
    if (tc::ld_acquire_gpu(cnt) >= target) return true;
    const long long t0 = clock64();
    while (true) {
        if (clock64() - t0 >= limit) return false;
        if (*abort) return false;
        __nanosleep(32);
        if (tc::ld_acquire_gpu(cnt) >= target) return true;
    }
}

// After a tile's stores: make them visible to the async proxy (TMA readers) and to other
// CTAs, then count the step done for this row tile.
__device__ __forceinline__ void tile_done(int32_t *cnt)
{
    tc::fence_proxy_async_global();
    tc::tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0) tc::red_release_gpu_add(cnt, 1);
}

template <int U>
__global__ void __launch_bounds__(kThreads, 1)
fwd_persist(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_h, PersistArgs p)
{
    constexpr int NB = 4 * U, NC = U / 8;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    const StepArgs &a = p.s;
    extern __shared__ uint8_t smem_raw[];
    __shared__ float s_bias[4 * U];
    const PCtl pc = pcarve(smem_raw, a.S, NB, a.KC, p.w_res);
    const Ctl &c = pc.c;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ct = blockIdx.x % p.n_ct, slot = blockIdx.x / p.n_ct, cl = p.cl;
    const uint32_t rank = cl > 1 ? tc::cluster_rank() : 0;
    const int B = a.B, H = a.H, kcx = a.kcx, KC = a.KC, S = a.S, T = a.T;
    const long long limit = a.limit;
    for (int i = tid; i < 4 * U; i += kThreads) {
        const int g = i / U, u = ct * U + i % U;
        s_bias[i] = u < H ? a.bias[g * H + u] : 0.0f;
    }
    const uint32_t tmem = pprologue(pc, S, kCols, cl);
    const uint8_t *wtile = a.wpack + (size_t)ct * KC * c.b_bytes;
    if (p.w_res && tid == 0) {
        tc::mbar_arrive_expect_tx(pc.wbar, KC * c.b_bytes);
        tc::bulk_g2s(pc.w0, wtile, KC * c.b_bytes, pc.wbar);
    }
    bool w_ready = !p.w_res;        // warp 0
    int n_issued = 0, n_waited = 0;  // warp 0: chunks armed / consumed (abort drain)

    // warp 0 (lane 0 issues): chunk it of tile (t, row0) into ring slot g, once every
    // CTA of the cluster drained the chunk that used the stage before
    auto produce = [&](int t, int row0, int it, uint32_t g) {
        const int s = (int)(g % S);
        if (g >= (uint32_t)S && !tc::mbar_wait(&c.empty[s], (g / S - 1) & 1, limit, c.abort)) {
            set_abort(c, a.err);
            return;
        }
        if (lane == 0) {
            const uint32_t bytes = kAStage + (p.w_res ? 0u : c.b_bytes);
            if (it < kcx)
                load_a_chunk(c, s, bytes, &tm_x, it * kChunk, t * B + row0, it, cl, rank);
            else
                load_a_chunk(c, s, bytes, &tm_h, (it - kcx) * kChunk, t * B + row0, it, cl, rank);
            if (!p.w_res) tc::bulk_g2s(c.b0 + s * c.b_bytes, wtile + (size_t)it * c.b_bytes, c.b_bytes, &c.full[s]);
        }
        __syncwarp();
        ++n_issued;
    };
    // warp 0 (lane 0 issues): MMAs of chunk it once its bytes landed
    auto consume = [&](int it, uint32_t g) {
        const int s = (int)(g % S);
        if (!w_ready) {
            if (!tc::mbar_wait(pc.wbar, 0, limit, c.abort)) {
                set_abort(c, a.err);
                return;
            }
            w_ready = true;
        }
        if (!tc::mbar_wait(&c.full[s], (g / S) & 1, limit, c.abort)) {
            set_abort(c, a.err);
            return;
        }
        ++n_waited;
        if (lane == 0) {
            tc::tc_fence_after();
            issue_kmajor<NB>(tmem, c.a0 + s * kAStage, p.w_res ? pc.w0 + it * c.b_bytes : c.b0 + s * c.b_bytes, it);
            commit_empty(&c.empty[s], cl);
        }
        __syncwarp();
    };

    // tiles in order: (t, rt) for t = 0.., rt = slot, slot + n_slot, ...
    int x_pre = 0;  // warp 0: x chunks of the coming tile already issued
    uint32_t gbase = 0, tiles = 0;
    bool stop = false;
    for (int t = 0; t < T && !stop; ++t) {
        for (int rt = slot; rt < p.n_rt; rt += p.n_slot) {
            const int row0 = rt * kRows, b = row0 + tid;
            const bool row_ok = b < B;
            const int src = row_ok ? a.top[(size_t)t * B + b] : 0;
            const int s_next = row_ok ? a.top[(size_t)(t + 1) * B + b] : 0;
            const bool is_new = s_next == t + 1;
            // operands this CTA wrote itself (same units): c_read, and the older top the
            // next step reads when step t does not push
            float cr[U];
            uint4 hc[NC];
#pragma unroll
            for (int cu = 0; cu < NC; ++cu) {
                const int u = ct * U + cu * 8;
                float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                hc[cu] = make_uint4(0, 0, 0, 0);
                if (row_ok && u < H) {
                    ld8f_cg(a.hist_c + ((size_t)src * B + b) * H + u, v);
                    if (!is_new) hc[cu] = __ldcg((const uint4 *)(a.hr + ((size_t)s_next * B + b) * H + u));
                }
#pragma unroll
                for (int e = 0; e < 8; ++e) cr[cu * 8 + e] = v[e];
            }
            if (warp == 0 && !*c.abort) {
                // one produce/consume loop: produce while the ring has room (chunk it needs
                // chunk it - S consumed), else consume. Chunks below x_pre were prefetched.
                // Before the first h chunk, wait until every column tile of this row tile
                // finished step t - 1 (they wrote hr[t]).
                bool dep_done = t == 0;
                for (int it = x_pre, jc = 0; jc < KC && !*c.abort;) {
                    if (it < KC && it - jc < S) {
                        if (it >= kcx && !dep_done) {
                            if (!spin_until(p.cnt + rt, p.n_ct * t, limit, c.abort)) set_abort(c, a.err);
                            tc::fence_proxy_async_global();
                            __syncwarp();
                            dep_done = true;
                            if (*c.abort) break;
                        }
                        produce(t, row0, it, gbase + it);
                        ++it;
                    } else {
                        consume(jc, gbase + jc);
                        ++jc;
                    }
                }
                if (lane == 0) tc::mma_commit(c.done);
                __syncwarp();
            }
            if (!tc::mbar_wait(c.done, tiles & 1, limit, nullptr)) {
                set_abort(c, a.err);
                tc::mbar_wait(c.done, tiles & 1, kDrainLimit, nullptr);
            }
            gbase += KC;
            ++tiles;
            __syncthreads();
            tc::tc_fence_after();
            if (*c.abort) {
                stop = true;
                break;
            }
            // prefetch the next tile's x chunks (the whole ring is free: this tile's MMAs are done)
            x_pre = 0;
            {
                int tn = t, rn = rt + p.n_slot;
                if (rn >= p.n_rt) {
                    rn = slot;
                    ++tn;
                }
                if (tn < T && warp == 0)
                    for (; x_pre < min(kcx, S) && !*c.abort; ++x_pre) produce(tn, rn * kRows, x_pre, gbase + x_pre);
            }
            const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
            for (int cu = 0; cu < NC; ++cu) {
                float z[4][8];
#pragma unroll
                for (int g = 0; g < 4; ++g) tc::tmem_ld8(trow + g * U + cu * 8, z[g]);
                const int u = ct * U + cu * 8;
                if (row_ok && u < H)
                    fwd_cell8(a, t, b, u, z, s_bias + cu * 8, s_bias + U + cu * 8, s_bias + 2 * U + cu * 8,
                              s_bias + 3 * U + cu * 8, cr + cu * 8, is_new, hc[cu]);
            }
            // hr[t + 1] is read by TMA: generic writes -> async proxy, then release the step
            tile_done(p.cnt + rt);
        }
    }
    if (warp == 0) {
        for (int jj = n_waited; jj < n_issued; ++jj) {  // chunks armed but not consumed (abort)
            const uint32_t g = (uint32_t)jj;
            tc::mbar_wait(&c.full[g % S], (g / S) & 1, kDrainLimit, nullptr);
        }
        if (!w_ready) tc::mbar_wait(pc.wbar, 0, kDrainLimit, nullptr);
    }
    if (cl > 1) tc::cluster_sync();  // nobody leaves while a peer may still multicast into it
    finish(c, tmem, kCols);
}

template <int U>
__global__ void __launch_bounds__(kThreads, 1) bwd_persist(const __grid_constant__ CUtensorMap tm_g, PersistArgs p)
{
    constexpr int NB = U, NC = U / 8;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    const StepArgs &a = p.s;
    extern __shared__ uint8_t smem_raw[];
    const PCtl pc = pcarve(smem_raw, a.S, NB, a.KC, p.w_res);
    const Ctl &c = pc.c;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ct = blockIdx.x % p.n_ct, slot = blockIdx.x / p.n_ct, cl = p.cl;
    const uint32_t rank = cl > 1 ? tc::cluster_rank() : 0;
    const int B = a.B, H = a.H, KC = a.KC, S = a.S, T = a.T;
    const long long limit = a.limit;
    const uint32_t tmem = pprologue(pc, S, kCols, cl);
    const uint8_t *wtile = a.wpack + (size_t)ct * KC * c.b_bytes;
    if (p.w_res && tid == 0) {
        tc::mbar_arrive_expect_tx(pc.wbar, KC * c.b_bytes);
        tc::bulk_g2s(pc.w0, wtile, KC * c.b_bytes, pc.wbar);
    }
    // the resident weight tile must land before the first MMA (warp 0, uniformly)
    if (p.w_res && warp == 0 && !tc::mbar_wait(pc.wbar, 0, limit, c.abort)) {
        set_abort(c, a.err);
        tc::mbar_wait(pc.wbar, 0, kDrainLimit, nullptr);
    }
    int n_issued = 0, n_waited = 0;
    uint32_t gbase = 0, tiles = 0;
    bool stop = false;
    for (int t = T - 1; t >= 0 && !stop; --t) {
        const int need = T - 1 - t;  // steps every column tile finished before this one
        for (int rt = slot; rt < p.n_rt; rt += p.n_slot) {
            const int row0 = rt * kRows, b = row0 + tid;
            const bool row_ok = b < B;
            const int src = row_ok ? a.top[(size_t)t * B + b] : 0;
            const int s1 = (row_ok && t >= 1) ? a.top[(size_t)(t - 1) * B + b] : 0;
            // Prefetch every epilogue operand: the gradient history of this CTA's units is
            // written only by this CTA; gates and cell states come from the forward.
            float dh_src[U], dh_t[U], dc_t[U], cn[U], cr[U], dc_rd[U];
            uint4 gq[NC][4];
#pragma unroll
            for (int cu = 0; cu < NC; ++cu) {
                const int u = ct * U + cu * 8;
                const bool ok = row_ok && u < H;
                float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                if (ok) ld8f_cg(a.dhist_h + ((size_t)src * B + b) * H + u, v);
#pragma unroll
                for (int e = 0; e < 8; ++e) dh_src[cu * 8 + e] = v[e];
                if (ok && t >= 1) {
                    const size_t wr = ((size_t)t * B + b) * H + u, rd = ((size_t)s1 * B + b) * H + u;
                    float w1[8], w2[8], w3[8], w4[8], w5[8];
                    ld8f_cg(a.dhist_h + wr, w1);
                    ld8f_cg(a.dhist_c + wr, w2);
                    ld8f_cg(a.hist_c + wr, w3);
                    ld8f_cg(a.hist_c + rd, w4);
                    ld8f_cg(a.dhist_c + rd, w5);
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        dh_t[cu * 8 + e] = w1[e]; dc_t[cu * 8 + e] = w2[e]; cn[cu * 8 + e] = w3[e];
                        cr[cu * 8 + e] = w4[e]; dc_rd[cu * 8 + e] = w5[e];
                    }
                    const __half *gt = a.gates + ((size_t)(t - 1) * B + b) * 4 * H + u;
#pragma unroll
                    for (int g = 0; g < 4; ++g) gq[cu][g] = *(const uint4 *)(gt + (size_t)g * H);
                }
            }
            if (warp == 0 && !*c.abort) {
                // dG_t was written at the previous step by every column tile of this row tile
                if (need > 0) {
                    if (!spin_until(p.cnt + rt, p.n_ct * need, limit, c.abort)) set_abort(c, a.err);
                    tc::fence_proxy_async_global();
                    __syncwarp();
                }
                for (int it = 0, jc = 0; jc < KC && !*c.abort;) {
                    if (it < KC && it - jc < S) {
                        const uint32_t g = gbase + it;
                        const int s = (int)(g % S);
                        if (g >= (uint32_t)S && !tc::mbar_wait(&c.empty[s], (g / S - 1) & 1, limit, c.abort)) {
                            set_abort(c, a.err);
                            break;
                        }
                        if (lane == 0) {
                            load_a_chunk(c, s, kAStage + (p.w_res ? 0u : c.b_bytes), &tm_g, it * kChunk, t * B + row0,
                                         it, cl, rank);
                            if (!p.w_res)
                                tc::bulk_g2s(c.b0 + s * c.b_bytes, wtile + (size_t)it * c.b_bytes, c.b_bytes,
                                             &c.full[s]);
                        }
                        __syncwarp();
                        ++n_issued;
                        ++it;
                    } else {
                        const uint32_t g = gbase + jc;
                        const int s = (int)(g % S);
                        if (!tc::mbar_wait(&c.full[s], (g / S) & 1, limit, c.abort)) {
                            set_abort(c, a.err);
                            break;
                        }
                        ++n_waited;
                        if (lane == 0) {
                            tc::tc_fence_after();
                            issue_kmajor<NB>(tmem, c.a0 + s * kAStage,
                                             p.w_res ? pc.w0 + jc * c.b_bytes : c.b0 + s * c.b_bytes, jc);
                            commit_empty(&c.empty[s], cl);
                        }
                        __syncwarp();
                        ++jc;
                    }
                }
                if (lane == 0) tc::mma_commit(c.done);
                __syncwarp();
            }
            if (!tc::mbar_wait(c.done, tiles & 1, limit, nullptr)) {
                set_abort(c, a.err);
                tc::mbar_wait(c.done, tiles & 1, kDrainLimit, nullptr);
            }
            gbase += KC;
            ++tiles;
            __syncthreads();
            tc::tc_fence_after();
            if (*c.abort) {
                stop = true;
                break;
            }
            if (need > 0) (void)tc::ld_acquire_gpu(p.cnt + rt);  // every thread: acquire before reading
            const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
            for (int cu = 0; cu < NC; ++cu) {
                float acc[8];
                tc::tmem_ld8(trow + cu * 8, acc);
                const int u = ct * U + cu * 8;
                if (row_ok && u < H) {
                    float v[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) v[e] = dh_src[cu * 8 + e] + acc[e];
                    st8f(a.dhist_h + ((size_t)src * B + b) * H + u, v);
                    if (t >= 1) {
                        float ig[8], fg[8], gg[8], og[8], d[4][8], dcr[8];
                        unpack8_f16(gq[cu][0], ig);
                        unpack8_f16(gq[cu][1], fg);
                        unpack8_f16(gq[cu][2], gg);
                        unpack8_f16(gq[cu][3], og);
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const int j = cu * 8 + e;
                            const float dh = src == t ? v[e] : dh_t[j];  // the state read at t is row t
                            const float tcn = tanh_hw(cn[j]);
                            const float dc = dc_t[j] + dh * og[e] * (1.0f - tcn * tcn);
                            d[0][e] = dc * gg[e] * ig[e] * (1.0f - ig[e]);
                            d[1][e] = dc * cr[j] * fg[e] * (1.0f - fg[e]);
                            d[2][e] = dc * ig[e] * (1.0f - gg[e] * gg[e]);
                            d[3][e] = dh * tcn * og[e] * (1.0f - og[e]);
                            dcr[e] = dc_rd[j] + dc * fg[e];
                        }
                        __nv_bfloat16 *dg = a.dG + ((size_t)(t - 1) * B + b) * 4 * H + u;
#pragma unroll
                        for (int g = 0; g < 4; ++g) *(uint4 *)(dg + (size_t)g * H) = pack8_bf16(d[g]);
                        st8f(a.dhist_c + ((size_t)s1 * B + b) * H + u, dcr);
                    }
                }
            }
            tile_done(p.cnt + rt);
        }
    }
    if (warp == 0)
        for (int jj = n_waited; jj < n_issued; ++jj) {  // chunks armed but not consumed (abort)
            const uint32_t g = (uint32_t)jj;
            tc::mbar_wait(&c.full[g % S], (g / S) & 1, kDrainLimit, nullptr);
        }
    if (cl > 1) tc::cluster_sync();  // nobody leaves while a peer may still multicast into it
    finish(c, tmem, kCols);
}

// ------------------------------------------------------------------ packing
// Forward operand: for column tile ct, rows n = g * U + j hold gate g of hidden unit
// ct * U + j; each row is the matching column of W over the contraction
// [x padded to 64 ; h padded to 64], in 64-element chunks of 128-byte swizzled rows.
__global__ void pack_fwd(const __nv_bfloat16 *__restrict__ W, int I, int H, int U, int kcx, int KC, int n_ct,
                         __nv_bfloat16 *__restrict__ out)
{
    const int NB = 4 * U, G = 4 * H;
    const size_t n = (size_t)n_ct * KC * NB * kChunk;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int col = (int)(e % kChunk);
        const size_t rowi = e / kChunk;  // (ct * KC + kc) * NB + row
        const int row = (int)(rowi % NB);
        const size_t tile = rowi / NB;
        const int kc = (int)(tile % KC), ct = (int)(tile / KC);
        const int g = row / U, unit = ct * U + row % U;
        int wrow = -1;
        if (kc < kcx) {
            const int k = kc * kChunk + col;
            if (k < I) wrow = k;
        } else {
            const int k = (kc - kcx) * kChunk + col;
            if (k < H) wrow = I + k;
        }
        const __nv_bfloat16 v =
            (unit < H && wrow >= 0) ? W[(size_t)wrow * G + g * H + unit] : __float2bfloat16(0.0f);
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
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encoder()
{
    if (g_encode) return cudaSuccess;
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess) return e;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    return cudaSuccess;
}

// Row-major bf16 matrix [rows][cols] read in boxes of 64 columns x box_rows rows with
// 128-byte swizzling; out-of-range elements read as zero.
cudaError_t make_map(void *slot, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows)
{
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)kChunk, box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = g_encode((CUtensorMap *)slot, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

enum { kMapX128 = 0, kMapX64 = 1, kMapG128 = 2, kMapG64 = 3, kMapH128 = 4, kMapH64 = 5 };
const CUtensorMap &map(const stacklstm *s, int i) { return *(const CUtensorMap *)s->tmaps[i]; }

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

constexpr uint32_t kSmemCap = 225 * 1024;

template <typename Kern>
cudaError_t allow_smem(Kern k)
{
    return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemCap);
}

// Ring depth: as many stages as the contraction has chunks, within a shared-memory
// budget that leaves room for two CTAs per SM when the grid needs more than one wave.
int pick_stages(int KC, int NB, size_t ctas, int sms)
{
    const uint32_t budget = ctas > (size_t)sms ? 100 * 1024 : 200 * 1024;
    const uint32_t stage = kAStage + (uint32_t)NB * 128;
    int S = (int)((budget - 1024 - (2 * kMaxStages + 1) * 8 - 16) / stage);
    return std::max(2, std::min({S, KC, kMaxStages}));
}

int pick_dx_n(int I) { return I <= 32 ? 32 : I <= 64 ? 64 : I <= 128 ? 128 : 256; }


// Plans a persistent launch. Column tiles may form thread-block clusters of cl CTAs that
// share their A chunks by multicast (the tile count is then padded to a multiple of cl;
// padding tiles hold zero weights and store nothing). Multicast pays only when the
// column tiles' re-reads of the A operand are a large L2 stream (want_mc); the cluster
// sizes tried are then 16, 8, 4, 2 and 1, else 1. For each size and shared-memory budget
// (one, two or three CTAs per SM) the weight tile stays resident when it leaves room for a
// ring of at least two stages, and the grid is sized from the number of co-resident
// clusters of that footprint. The fewest row tiles per CTA per step wins; ties go to the
// larger cluster, then the deeper ring. Returns false if nothing fits.
template <typename Kern>
bool plan_persist(Kern kernel, int KC, int NB, int n_ct, int n_rt, bool want_mc, int *slot, int *wres, int *S,
                  int *cl, int *nct_pad)
{
    const uint32_t fixed = 1024 + (2 * kMaxStages + 2) * 8 + 16 + 1024 /* static */;
    const uint32_t wbytes = (uint32_t)KC * NB * 128;
    int best_rounds = 1 << 30, best_c = 0;
    bool found = false;
    for (int c : {16, 8, 4, 2, 1}) {
        if (c > 1 && (!want_mc || c / 2 >= n_ct)) continue;
        const int pad = (n_ct + c - 1) / c * c;
        if (c > 8 && cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        for (uint32_t budget : {200u * 1024, 100u * 1024, 66u * 1024}) {
            const int wr = wbytes + 2 * kAStage + fixed <= budget;
            const uint32_t stage = kAStage + (wr ? 0u : (uint32_t)NB * 128);
            if (budget < fixed + (wr ? wbytes : 0u) + 2 * stage) continue;
            const int st =
                std::max(2, std::min({(int)((budget - fixed - (wr ? wbytes : 0u)) / stage), KC, kMaxStages}));
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(pad);
            cfg.blockDim = dim3(kThreads);
            cfg.dynamicSmemBytes = psmem_bytes(st, NB, KC, wr);
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = c;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            cfg.attrs = at;
            cfg.numAttrs = 1;
            int clusters = 0;
            if (cudaOccupancyMaxActiveClusters(&clusters, kernel, &cfg) != cudaSuccess) {
                cudaGetLastError();
                continue;
            }
            const int groups = pad / c;  // clusters that cover the column tiles once
            if (clusters < groups) continue;
            const int sl = std::min(n_rt, clusters / groups);
            const int rounds = (n_rt + sl - 1) / sl;
            if (rounds < best_rounds || (rounds == best_rounds && c > best_c)) {
                best_rounds = rounds;
                best_c = c;
                *slot = sl;
                *wres = wr;
                *S = st;
                *cl = c;
                *nct_pad = pad;
                found = true;
            }
        }
    }
    return found;
}

// Cooperative (all CTAs co-resident) cluster launch of a persistent kernel.
template <typename Kern, typename... Args>
cudaError_t launch_persist(Kern kernel, dim3 grid, size_t smem, cudaStream_t st, int cl, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeCooperative;
    at[0].val.cooperative = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cl;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

unsigned grid_for(const stacklstm *s, size_t n)
{
    return (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 16));
}

StepArgs step_args(stacklstm *s, const float *bias, const void *wpack, int kcx, int KC, int S)
{
    StepArgs a;
    a.T = s->T; a.B = s->B; a.I = s->I; a.H = s->H;
    a.kcx = kcx; a.KC = KC; a.S = S;
    a.top = s->top;
    a.hist_h = (__nv_bfloat16 *)s->hist_h; a.hr = (__nv_bfloat16 *)s->hr;
    a.hist_c = s->hist_c; a.gates = (__half *)s->gates;
    a.bias = bias; a.wpack = (const uint8_t *)wpack;
    a.dhist_h = s->dhist_h; a.dhist_c = s->dhist_c; a.dG = (__nv_bfloat16 *)s->dG;
    a.limit = s->wait_limit; a.err = s->err;
    return a;
}

}  // namespace

std::string bf16_describe(const stacklstm *s)
{
    char buf[512];
    const int rt = (int)ceil_div(s->B, kRows);
    snprintf(buf, sizeof buf,
             "bf16 tcgen05; row tiles %d; forward %s U=%d chunks %d (x %d)%s; backward %s U=%d chunks %d; "
             "persistent fwd: slots %d cluster %d col tiles %d ring %d w_res %d; persistent bwd: slots %d cluster %d "
             "col tiles %d ring %d w_res %d; step rings fwd %d bwd %d; dx N=%d x%d ring %d; dW %dx%d tiles x%d "
             "splits ring %d",
             rt, s->pf ? "persistent" : "per-step", s->uf, s->kcf, s->kcx, "", s->pb ? "persistent" : "per-step",
             s->ub, s->kcb, s->pf_slot, s->pf_cl, s->pf_nct, s->pf_S, s->pf_wres, s->pb_slot, s->pb_cl, s->pb_nct,
             s->pb_S, s->pb_wres, s->sf, s->sb, s->nx, s->nxt, s->sx, s->dw_mt, s->dw_nt, s->dw_split, s->sw);
    return buf;
}

const char *bf16_unsupported(int T, int B, int I, int H)
{
    if (I % 8 || H % 8) return "bf16 path needs I and H to be multiples of 8";
    if ((long long)T * B >= (1LL << 31) - 256) return "T * B too large for 32-bit tensor coordinates";
    return nullptr;
}

cudaError_t bf16_prepare(stacklstm *s)
{
    cudaError_t e;
    if ((e = get_encoder())) return e;
    const int T = s->T, B = s->B, I = s->I, H = s->H, rt = (int)ceil_div(B, kRows), sms = s->num_sms;
    s->uf = (int)ceil_div(H, 32) * rt >= sms ? 32 : (int)ceil_div(H, 16) * rt >= sms / 2 ? 16 : 8;
    s->ub = (int)ceil_div(H, 32) * rt >= sms ? 32 : 16;
    s->kcx = (int)ceil_div(I, kChunk);
    s->kcf = s->kcx + (int)ceil_div(H, kChunk);
    s->kcb = (int)ceil_div(4 * H, kChunk);
    s->nx = pick_dx_n(I);
    s->nxt = (int)ceil_div(I, s->nx);
    s->dw_mt = (int)ceil_div(I + H + 1, kRows);
    s->dw_nt = (int)ceil_div(4 * H, 256);
    const size_t R = (size_t)T * B, RC = ceil_div(R, kChunk);
    s->dw_split = (int)std::max<size_t>(1, std::min<size_t>(sms / std::max(1, s->dw_mt * s->dw_nt), RC / 2));
    const char *lim = getenv("STACKLSTM_WAIT_LIMIT_CYCLES");
    s->wait_limit = lim ? atoll(lim) : 4000000000LL;
    if ((e = allow_smem(fwd_persist<32>)) || (e = allow_smem(fwd_persist<16>)) || (e = allow_smem(fwd_persist<8>)) ||
        (e = allow_smem(bwd_persist<16>)) || (e = allow_smem(fwd_step_tc<32>)) ||
        (e = allow_smem(fwd_step_tc<16>)) || (e = allow_smem(fwd_step_tc<8>)) || (e = allow_smem(bwd_step_tc<32>)) ||
        (e = allow_smem(bwd_step_tc<16>)) || (e = allow_smem(dx_tc<32>)) || (e = allow_smem(dx_tc<64>)) ||
        (e = allow_smem(dx_tc<128>)) || (e = allow_smem(dx_tc<256>)) || (e = allow_smem(dw_tc)))
        return e;

    // persistent step kernels unless disabled (STACKLSTM_STEP_KERNELS=1 keeps one launch per step)
    const char *per_step = getenv("STACKLSTM_STEP_KERNELS");
    if (!(per_step && atoi(per_step) != 0)) {
        // A-operand bytes the column tiles re-read from L2 per step without multicast
        const int nctf = (int)ceil_div(H, s->uf), nctb16 = (int)ceil_div(H, 16);
        // multicast clusters measured slower than independent CTAs on every workload tried
        // so far; STACKLSTM_MULTICAST=1 enables them where the re-read stream is large
        const char *mc = getenv("STACKLSTM_MULTICAST");
        const bool mc_on = mc && atoi(mc) != 0;
        const bool mcf = mc_on && (double)rt * kAStage * s->kcf * nctf >= 8e6;
        const bool mcb = mc_on && (double)rt * kAStage * s->kcb * nctb16 >= 8e6;
        if (s->uf == 32)
            s->pf = plan_persist(fwd_persist<32>, s->kcf, 128, nctf, rt, mcf, &s->pf_slot, &s->pf_wres, &s->pf_S,
                                 &s->pf_cl, &s->pf_nct);
        else if (s->uf == 16)
            s->pf = plan_persist(fwd_persist<16>, s->kcf, 64, nctf, rt, mcf, &s->pf_slot, &s->pf_wres, &s->pf_S,
                                 &s->pf_cl, &s->pf_nct);
        else
            s->pf = plan_persist(fwd_persist<8>, s->kcf, 32, nctf, rt, mcf, &s->pf_slot, &s->pf_wres, &s->pf_S,
                                 &s->pf_cl, &s->pf_nct);
        // the persistent backward keeps 16-unit tiles (its prefetched epilogue operands
        // need the registers); the weight packing follows
        s->pb = plan_persist(bwd_persist<16>, s->kcb, 16, nctb16, rt, mcb, &s->pb_slot, &s->pb_wres,
                             &s->pb_S, &s->pb_cl, &s->pb_nct);
        if (s->pb) s->ub = 16;
    }
    s->sf = pick_stages(s->kcf, 4 * s->uf, ceil_div(H, s->uf) * (size_t)rt, sms);
    s->sb = pick_stages(s->kcb, s->ub, ceil_div(H, s->ub) * (size_t)rt, sms);
    s->sx = pick_stages(s->kcb, s->nx, s->nxt * ceil_div(R, kRows), sms);
    s->sw = pick_stages((int)ceil_div(RC, s->dw_split), 256, (size_t)s->dw_mt * s->dw_nt * s->dw_split, sms);

    const size_t fwd_bytes = (size_t)std::max<size_t>(ceil_div(H, s->uf), s->pf ? s->pf_nct : 0) * s->kcf * 4 *
                             s->uf * 128;
    const size_t bwd_bytes = (size_t)std::max<size_t>(ceil_div(H, s->ub), s->pb ? s->pb_nct : 0) * s->kcb * s->ub *
                             128;
    const size_t dx_bytes = (size_t)s->nxt * s->kcb * s->nx * 128;
    s->dw_part_elems = (size_t)s->dw_split * s->dw_mt * kRows * s->dw_nt * 256;
    void *p;
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
    if (s->pf || s->pb) {
        if ((e = cudaMalloc(&p, 2 * sizeof(int32_t) * rt))) return e;
        s->allocs.push_back(p);
        s->rowcnt = (int32_t *)p;
    }
    // dG is workspace: its tensor maps are fixed for the handle's lifetime
    if ((e = make_map(s->tmaps[kMapG128], s->dG, R, 4 * (uint64_t)H, kRows))) return e;
    if ((e = make_map(s->tmaps[kMapG64], s->dG, R, 4 * (uint64_t)H, kChunk))) return e;
    const uint64_t R1 = (uint64_t)(T + 1) * B;
    if ((e = make_map(s->tmaps[kMapH128], s->hr, R1, (uint64_t)H, kRows))) return e;
    if ((e = make_map(s->tmaps[kMapH64], s->hr, R1, (uint64_t)H, kChunk))) return e;
    return cudaSuccess;
}

cudaError_t bf16_forward(stacklstm *s, const __nv_bfloat16 *x, const __nv_bfloat16 *h0, const float *c0,
                         const __nv_bfloat16 *W, const float *bias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H;
    cudaError_t e;
    s->x_saved = x;
    if ((e = make_map(s->tmaps[kMapX128], x, (uint64_t)T * B, I, kRows))) return e;
    if ((e = make_map(s->tmaps[kMapX64], x, (uint64_t)T * B, I, kChunk))) return e;
    if ((e = cudaMemcpyAsync(s->hist_h, h0, sizeof(__nv_bfloat16) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return e;
    if ((e = cudaMemcpyAsync(s->hr, h0, sizeof(__nv_bfloat16) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return e;
    if ((e = cudaMemcpyAsync(s->hist_c, c0, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream))) return e;
    const int nctf = std::max((int)ceil_div(H, s->uf), s->pf ? s->pf_nct : 0);
    const int nctb = std::max((int)ceil_div(H, s->ub), s->pb ? s->pb_nct : 0);
    pack_fwd<<<grid_for(s, (size_t)nctf * s->kcf * 4 * s->uf * kChunk), 256, 0, s->stream>>>(
        W, I, H, s->uf, s->kcx, s->kcf, nctf, (__nv_bfloat16 *)s->w_fwd);
    pack_rows<<<grid_for(s, (size_t)nctb * s->kcb * s->ub * kChunk), 256, 0, s->stream>>>(
        W, H, I, H, s->ub, s->kcb, nctb, (__nv_bfloat16 *)s->w_bwd);
    pack_rows<<<grid_for(s, (size_t)s->nxt * s->kcb * s->nx * kChunk), 256, 0, s->stream>>>(
        W, H, 0, I, s->nx, s->kcb, s->nxt, (__nv_bfloat16 *)s->w_dx);
    s->launches += 3;
    if ((e = cudaGetLastError())) return e;
    if (s->pf) {
        PersistArgs p;
        p.s = step_args(s, bias, s->w_fwd, s->kcx, s->kcf, s->pf_S);
        p.n_ct = s->pf_nct; p.n_rt = (int)ceil_div(B, kRows); p.n_slot = s->pf_slot; p.w_res = s->pf_wres;
        p.cl = s->pf_cl; p.cnt = s->rowcnt;
        if ((e = cudaMemsetAsync(p.cnt, 0, sizeof(int32_t) * p.n_rt, s->stream))) return e;
        const dim3 g(p.n_ct * p.n_slot);
        const size_t sm = psmem_bytes(p.s.S, 4 * s->uf, s->kcf, p.w_res);
        const CUtensorMap &tm = map(s, kMapX128), &th = map(s, kMapH128);
        if (s->uf == 32)
            e = launch_persist(fwd_persist<32>, g, sm, s->stream, p.cl, tm, th, p);
        else if (s->uf == 16)
            e = launch_persist(fwd_persist<16>, g, sm, s->stream, p.cl, tm, th, p);
        else
            e = launch_persist(fwd_persist<8>, g, sm, s->stream, p.cl, tm, th, p);
        if (e) return e;
        s->launches += 1;
        return cudaGetLastError();
    }
    const StepArgs a = step_args(s, bias, s->w_fwd, s->kcx, s->kcf, s->sf);
    const dim3 grid(nctf, ceil_div(B, kRows));
    const size_t smem = smem_bytes(s->sf, 4 * s->uf);
    const CUtensorMap &tmx = map(s, kMapX128), &tmh = map(s, kMapH128);
    for (int t = 0; t < T; ++t) {
        const bool pdl = t > 0;
        if (s->uf == 32)
            e = launch(fwd_step_tc<32>, grid, smem, s->stream, pdl, tmx, tmh, a, t);
        else if (s->uf == 16)
            e = launch(fwd_step_tc<16>, grid, smem, s->stream, pdl, tmx, tmh, a, t);
        else
            e = launch(fwd_step_tc<8>, grid, smem, s->stream, pdl, tmx, tmh, a, t);
        if (e) return e;
        s->launches += 1;
    }
    return cudaGetLastError();
}

cudaError_t bf16_backward_steps(stacklstm *s)
{
    const int T = s->T, B = s->B, H = s->H;
    cudaError_t e;
    const StepArgs a = step_args(s, nullptr, s->w_bwd, 0, s->kcb, s->sb);
    pointwise_last<<<grid_for(s, (size_t)B * (H / 8)), 256, 0, s->stream>>>(a);
    s->launches += 1;
    if ((e = cudaGetLastError())) return e;
    if (s->pb) {
        PersistArgs p;
        p.s = step_args(s, nullptr, s->w_bwd, 0, s->kcb, s->pb_S);
        p.n_ct = s->pb_nct; p.n_rt = (int)ceil_div(B, kRows); p.n_slot = s->pb_slot;
        p.w_res = s->pb_wres; p.cl = s->pb_cl; p.cnt = s->rowcnt + p.n_rt;
        if ((e = cudaMemsetAsync(p.cnt, 0, sizeof(int32_t) * p.n_rt, s->stream))) return e;
        const dim3 g(p.n_ct * p.n_slot);
        const size_t sm = psmem_bytes(p.s.S, s->ub, s->kcb, p.w_res);
        const CUtensorMap &tm = map(s, kMapG128);
        e = launch_persist(bwd_persist<16>, g, sm, s->stream, p.cl, tm, p);
        if (e) return e;
        s->launches += 1;
        return cudaGetLastError();
    }
    const dim3 grid(ceil_div(H, s->ub), ceil_div(B, kRows));
    const size_t smem = smem_bytes(s->sb, s->ub);
    const CUtensorMap &tmg = map(s, kMapG128);
    for (int t = T - 1; t >= 0; --t) {
        const bool pdl = t < T - 1;
        if (s->ub == 32)
            e = launch(bwd_step_tc<32>, grid, smem, s->stream, pdl, tmg, a, t);
        else
            e = launch(bwd_step_tc<16>, grid, smem, s->stream, pdl, tmg, a, t);
        if (e) return e;
        s->launches += 1;
    }
    return cudaGetLastError();
}

cudaError_t bf16_dx(stacklstm *s, float *dx)
{
    if (!dx) return cudaSuccess;
    const size_t R = (size_t)s->T * s->B;
    DxArgs d;
    d.R = R; d.I = s->I; d.KC = s->kcb; d.S = s->sx;
    d.wpack = (const uint8_t *)s->w_dx; d.dx = dx; d.limit = s->wait_limit; d.err = s->err;
    const dim3 g(s->nxt, ceil_div(R, kRows));
    const size_t smem = smem_bytes(s->sx, s->nx);
    const CUtensorMap &tmg = map(s, kMapG128);
    cudaError_t e;
    switch (s->nx) {
    case 32: e = launch(dx_tc<32>, g, smem, s->stream, false, tmg, d); break;
    case 64: e = launch(dx_tc<64>, g, smem, s->stream, false, tmg, d); break;
    case 128: e = launch(dx_tc<128>, g, smem, s->stream, false, tmg, d); break;
    default: e = launch(dx_tc<256>, g, smem, s->stream, false, tmg, d); break;
    }
    if (e) return e;
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t bf16_dw(stacklstm *s, float *dW, float *dbias)
{
    if (!dW && !dbias) return cudaSuccess;
    const int T = s->T, B = s->B, I = s->I, H = s->H;
    DwArgs w;
    w.B = B; w.I = I; w.H = H;
    w.x = (const __nv_bfloat16 *)s->x_saved; w.hr = (const __nv_bfloat16 *)s->hr;
    w.ones = (const __nv_bfloat16 *)s->ones;
    w.R = T * B; w.n_tiles_n = s->dw_nt; w.split = s->dw_split; w.S = s->sw; w.part = s->dw_part;
    w.ld_part = (size_t)s->dw_nt * 256; w.rows_part = (size_t)s->dw_mt * kRows;
    w.limit = s->wait_limit; w.err = s->err;
    cudaError_t e = launch(dw_tc, dim3(s->dw_mt * s->dw_nt, s->dw_split), smem_bytes(s->sw, 256), s->stream, false,
                           map(s, kMapX64), map(s, kMapH64), map(s, kMapG64), w);
    if (e) return e;
    dw_reduce<<<grid_for(s, (size_t)(I + H + 1) * 4 * H), 256, 0, s->stream>>>(
        I + H, 4 * H, s->dw_split, s->dw_part, w.rows_part, w.ld_part, dW, dbias);
    s->launches += 2;
    return cudaGetLastError();
}

}  // namespace sl
