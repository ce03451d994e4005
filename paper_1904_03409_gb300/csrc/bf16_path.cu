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
// After the loop: dx = dG W_x^T (one K-major contraction over all T*B rows); dW and dbias
// are in bf16_dw.cu. The persistent (one launch for all steps) versions of the step
// kernels are in bf16_persist.cu.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <stdio.h>
#include <stdlib.h>

#include <algorithm>

#include "bf16_dev.cuh"

namespace sl {
namespace {


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
    // gate g of unit u: row-major [T][B][4H], or blocked [T][B][H / 16][4][16]
    const size_t gs = a.gates_blk ? 16 : (size_t)H;
    const __half *gt = a.gates_blk ? a.gates + (((size_t)tp * B + b) * ((H + 15) / 16) + u / 16) * 64 + u % 16
                                   : a.gates + ((size_t)tp * B + b) * 4 * H + u;
    unpack8_f16(*(const uint4 *)(gt), ig);
    unpack8_f16(*(const uint4 *)(gt + gs), fg);
    unpack8_f16(*(const uint4 *)(gt + 2 * gs), gg);
    unpack8_f16(*(const uint4 *)(gt + 3 * gs), og);
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

// Pointwise backward of the last step (t = T - 1), before the reverse loop. With d_top_h
// (and no per-step dy) it first adds the loss gradient of the final top to that state's
// gradient-history row, ftop[b] (the seeding, done by the thread that owns the elements).
__global__ void pointwise_last(StepArgs a, const float *__restrict__ d_top_h, const int32_t *__restrict__ ftop)
{
    const int groups = a.H / 8;
    const size_t n = (size_t)a.B * groups;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(e / groups), u = (int)(e - (size_t)b * groups) * 8;
        if (d_top_h) {
            float *row = a.dhist_h + ((size_t)ftop[b] * a.B + b) * a.H + u;
            float acc[8], sd[8];
            ld8f_cg(row, acc);
            ld8f_cg(d_top_h + (size_t)b * a.H + u, sd);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] += sd[i];
            st8f(row, acc);
        }
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
    const int32_t *xidx;  // push-only mode: real step of each virtual row's step (-1: none), else null
    int B;
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
    // split contraction (grid z > 1): part z takes chunks [kc0, kc1) and writes its partial
    // product to slab z of the output
    const int kz = blockIdx.z, nz = gridDim.z;
    const int kc0 = (int)((long long)a.KC * kz / nz), kc1 = (int)((long long)a.KC * (kz + 1) / nz);
    float *out = a.dx + (size_t)kz * a.R * a.I;
    const uint8_t *bpack = a.wpack + ((size_t)ct * a.KC + kc0) * c.b_bytes;
    auto tma = [&](int it, int s, uint64_t *bar) {
        tc::mbar_arrive_expect_tx(bar, kAStage + c.b_bytes);
        tc::tma_load_2d(c.a0 + s * kAStage, &tm_g, (kc0 + it) * kChunk, (int)row0, bar);
        tc::bulk_g2s(c.b0 + s * c.b_bytes, bpack + (size_t)it * c.b_bytes, c.b_bytes, bar);
    };
    auto no_gather = [](int, int) {};
    auto issue = [&](int s, int j) { issue_kmajor<N>(tmem, c.a0 + s * kAStage, c.b0 + s * c.b_bytes, j); };
    mainloop<false>(c, a.S, kc1 - kc0, -1, a.limit, a.err, tma, no_gather, issue);
    if (!*c.abort) {
        const size_t row = row0 + tid;
        // the dx row this accumulator row belongs to: the same row, or (push-only mode)
        // the real step of this virtual row's push; rows past an instance's pushes have none
        bool ok_row = row < a.R;
        size_t orow = row;
        if (ok_row && a.xidx) {
            const int t = a.xidx[row];
            ok_row = t >= 0;
            orow = (size_t)t * a.B + row % a.B;
        }
        const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
        for (int cu = 0; cu < N / 8; ++cu) {
            float v[8];
            tc::tmem_ld8(trow + cu * 8, v);
            const int col = ct * N + cu * 8;
            if (ok_row && col < a.I) st8f(out + orow * a.I + col, v);
        }
    }
    finish(c, tmem, kCols);
}

// ------------------------------------------------------------------ packing
// The forward setup in one launch: the initial state into history row 0 (h0 also as the
// first h operand) and every weight tile the launches that follow read, each job a range of
// a flat element index (pack_*_elem, bf16_dev.cuh).
struct SetupArgs {
    const __nv_bfloat16 *W;
    int I, H;
    __nv_bfloat16 *wf;  // forward gate columns (n_f elements; 0: packed elsewhere)
    int uf, kcx, kcf;
    __nv_bfloat16 *wb;  // persistent / per-step backward rows (n_b; 0: not needed)
    int ub, kcb;
    __nv_bfloat16 *wdx;  // input-gradient rows (n_dx)
    int nx;
    __nv_bfloat16 *wcl;  // cluster backward slices (n_cl; 0: not needed)
    int n_ctc;
    const uint4 *h0, *c0;  // 16-byte pieces: n_h of h0, n_c of c0
    uint4 *hist_h, *hr, *hist_c;
    size_t n_f, n_b, n_dx, n_cl, n_h, n_c;
};

__global__ void setup_kernel(SetupArgs a)
{
    const size_t n = a.n_h + a.n_c + a.n_f + a.n_b + a.n_dx + a.n_cl;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        size_t r = e;
        if (r < a.n_h) {
            const uint4 v = a.h0[r];
            a.hist_h[r] = v;
            a.hr[r] = v;
            continue;
        }
        if ((r -= a.n_h) < a.n_c) {
            a.hist_c[r] = a.c0[r];
            continue;
        }
        if ((r -= a.n_c) < a.n_f) {
            pack_gate_cols_elem(r, a.W, a.I, a.H, a.uf, a.kcx, a.kcf, a.wf);
            continue;
        }
        if ((r -= a.n_f) < a.n_b) {
            pack_w_rows_elem(r, a.W, a.H, a.I, a.H, a.ub, a.kcb, a.wb);
            continue;
        }
        if ((r -= a.n_b) < a.n_dx) {
            pack_w_rows_elem(r, a.W, a.H, 0, a.I, a.nx, a.kcb, a.wdx);
            continue;
        }
        pack_bwd_slice_elem(r - a.n_dx, a.W, a.I, a.H, a.n_ctc, a.wcl);
    }
}

// Push-only mode: the input of each virtual step, x_push[k][b] = x[xidx[k][b]][b] (zero
// rows past the instance's pushes), 16-byte pieces (I % 8 == 0), one a thread. IDX is the
// index type: 32-bit whenever the pieces number fewer than 2^32 (its divisions are a
// fraction of the 64-bit ones).
template <typename IDX>
__global__ void gather_push_x(IDX rows, IDX B, IDX I8, const int32_t *__restrict__ xidx, const uint4 *__restrict__ x,
                              uint4 *__restrict__ out)
{
    const IDX n = rows * I8;
    for (IDX e = blockIdx.x * (IDX)blockDim.x + threadIdx.x; e < n; e += (IDX)gridDim.x * blockDim.x) {
        const IDX r = e / I8;
        const int t = xidx[r];
        out[e] = t >= 0 ? x[((size_t)t * B + r % B) * I8 + (e - r * I8)] : make_uint4(0u, 0u, 0u, 0u);
    }
}

// Generic K-major operand tiles [n tiles][KC][NB rows][64], 128-byte swizzled rows: row n
// of the operand is src row n (trans = false: src[n][k]) or src column n (trans = true:
// src[k][n]), zero past N and K.
__global__ void pack_kmajor(const __nv_bfloat16 *__restrict__ src, size_t ld, int trans, int N, int K, int NB, int KC,
                            int n_tiles, __nv_bfloat16 *__restrict__ out)
{
    const size_t n_el = (size_t)n_tiles * KC * NB * kChunk;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n_el; e += (size_t)gridDim.x * blockDim.x) {
        const int col = (int)(e % kChunk);
        const size_t rowi = e / kChunk;
        const int row = (int)(rowi % NB);
        const size_t tile = rowi / NB;
        const int kc = (int)(tile % KC), nt = (int)(tile / KC);
        const int n = nt * NB + row, k = kc * kChunk + col;
        __nv_bfloat16 v = __float2bfloat16(0.0f);
        if (n < N && k < K) v = trans ? src[(size_t)k * ld + n] : src[(size_t)n * ld + k];
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

// Row-major bf16 matrix [rows][cols] (rows `ld` elements apart, ld = cols unless given)
// read in boxes of 64 columns x box_rows rows with 128-byte swizzling; out-of-range
// elements read as zero.
cudaError_t make_map(void *slot, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows, uint64_t ld = 0)
{
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {(ld ? ld : cols) * 2};
    cuuint32_t box[2] = {(cuuint32_t)kChunk, box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = g_encode((CUtensorMap *)slot, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Swizzle mode of a staging tile whose rows are `bytes` long (16 to 128): the forward's
// epilogue writes its staging tiles in this layout.
CUtensorMapSwizzle stage_swizzle(uint32_t bytes)
{
    return bytes >= 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                        : bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                      : bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B : CU_TENSOR_MAP_SWIZZLE_NONE;
}

// The saved gates [T][B][4][H] (fp16) as a 4-D tensor for the forward's tensor stores:
// boxes of `units` hidden units x 1 gate x rows instances x 1 step, so a store never
// writes past H (into the next gate) or past B (into the next step).
cudaError_t make_gates_map(void *slot, const void *base, int T, int B, int H, uint32_t units)
{
    cuuint64_t dims[4] = {(cuuint64_t)H, 4, (cuuint64_t)B, (cuuint64_t)T};
    cuuint64_t strides[3] = {(cuuint64_t)H * 2, (cuuint64_t)H * 8, (cuuint64_t)H * 8 * B};
    cuuint32_t box[4] = {units, 1, (cuuint32_t)std::min(B, kRows), 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = g_encode((CUtensorMap *)slot, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void *>(base), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, stage_swizzle(units * 2),
                          CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// The history rows h' [T+1][B][H] (bf16) or c' (fp32) as a 3-D tensor for the forward's
// tensor stores: boxes of `units` hidden units x rows instances x 1 step.
cudaError_t make_hist_map(void *slot, const void *base, bool fp32, int T, int B, int H, uint32_t units)
{
    const cuuint64_t es = fp32 ? 4 : 2;
    cuuint64_t dims[3] = {(cuuint64_t)H, (cuuint64_t)B, (cuuint64_t)T + 1};
    cuuint64_t strides[2] = {(cuuint64_t)H * es, (cuuint64_t)H * es * B};
    cuuint32_t box[3] = {units, (cuuint32_t)std::min(B, kRows), 1};
    cuuint32_t el[3] = {1, 1, 1};
    CUresult r = g_encode((CUtensorMap *)slot, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                          3, const_cast<void *>(base), dims, strides, box, el, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          stage_swizzle(units * (uint32_t)es), CU_TENSOR_MAP_L2_PROMOTION_NONE,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

enum { kMapX128 = 0, kMapX64 = 1, kMapG128 = 2, kMapG64 = 3, kMapH128 = 4, kMapH64 = 5, kMapGates = 6, kMapHistH = 7,
       kMapHistC = 8 };
const CUtensorMap &map(const stacklstm *s, int i) { return *(const CUtensorMap *)s->tmaps[i]; }

// budget that leaves room for two CTAs per SM when the grid needs more than one wave.
int pick_stages(int KC, int NB, size_t ctas, int sms)
{
    const uint32_t budget = ctas > (size_t)sms ? 100 * 1024 : 200 * 1024;
    const uint32_t stage = kAStage + (uint32_t)NB * 128;
    int S = (int)((budget - 1024 - (2 * kMaxStages + 1) * 8 - 16) / stage);
    return std::max(2, std::min({S, KC, kMaxStages}));
}

int pick_dx_n(int I) { return I <= 32 ? 32 : I <= 64 ? 64 : I <= 128 ? 128 : 256; }


unsigned grid_for(const stacklstm *s, size_t n)
{
    return (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 16));
}

StepArgs step_args(stacklstm *s, const float *bias, const void *wpack, int kcx, int KC, int S)
{
    StepArgs a;
    // the step kernels run over s->Tr steps: the real ones, or (push-only mode) the
    // virtual timeline of each instance's pushes with its own read indices
    a.T = s->Tr; a.B = s->B; a.I = s->I; a.H = s->H;
    a.kcx = kcx; a.KC = KC; a.S = S;
    a.top = s->push_only ? s->vtop : s->top;
    a.hist_h = (__nv_bfloat16 *)s->hist_h; a.hr = (__nv_bfloat16 *)s->hr;
    a.hist_c = s->hist_c; a.gates = (__half *)s->gates; a.gates_blk = 0;
    a.bias = bias; a.wpack = (const uint8_t *)wpack;
    a.dhist_h = s->dhist_h; a.dhist_c = s->dhist_c; a.dG = (__nv_bfloat16 *)s->dG;
    a.limit = s->wait_limit; a.err = s->err;
    return a;
}
// the backward's step arguments: as step_args, with the backward's wait budget
StepArgs bwd_args(stacklstm *s, const void *wpack, int KC, int S)
{
    StepArgs a = step_args(s, nullptr, wpack, 0, KC, S);
    a.limit = s->wait_limit_bwd;
    return a;
}

}  // namespace

std::string bf16_describe(const stacklstm *s)
{
    char buf[1024];
    const int rt = (int)ceil_div(s->B, kRows);
    const PersistPlan &f = s->cc.on ? s->cc : s->fc.on ? s->fc : s->pf, &b = s->cc.on ? s->cc : s->bc.on ? s->bc : s->pb;
    snprintf(buf, sizeof buf,
             "bf16 tcgen05; row tiles %d; chunks fwd %d (x %d) bwd %d; "
             "forward %s U=%d [EP %d G %d ring %d slots %d cluster %d col tiles %d w_res %d smem %u threads %d "
             "per SM %d]; "
             "backward %s U=%d [EP %d G %d ring %d slots %d cluster %d col tiles %d w_res %d smem %u threads %d "
             "per SM %d "
             "contraction parts %d dx CTAs %d ring %d]; "
             "step rings fwd %d bwd %d; dx N=%d x%d ring %d; dW %dx%d tiles of %dx%d x%d splits ring %d",
             rt, s->kcf, s->kcx, s->kcb, s->cc.on ? "cuda-core" : s->fc.on ? "cluster" : f.on ? "persistent" : "per-step", s->uf, f.EP, f.G, f.S, f.slot, f.cl, f.n_ct,
             f.w_res, f.smem, f.threads, f.per_sm, s->cc.on ? "cuda-core" : s->bc.on ? "cluster" : b.on ? "persistent" : "per-step", s->bc.on ? s->bc.U : s->ub, b.EP, b.G, b.S, b.slot, b.cl, b.n_ct,
             b.w_res, b.smem, b.threads, b.per_sm, b.KS, b.n_dx, b.dx_S, s->sf, s->sb, s->nx, s->nxt, s->sx, s->dw_mt, s->dw_nt, s->dw_mtile, s->dw_ntile, s->dw_split, s->sw);
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
    const size_t R = (size_t)T * B;
    // test hook (include/stacklstm.h): the clock budget of one device-side wait
    const char *lim = getenv("STACKLSTM_WAIT_LIMIT_CYCLES");
    s->wait_limit = lim ? atoll(lim) : 4000000000LL;
    // test hook: the backward's kernels alone (so that a forward can run before they time out)
    const char *limb = getenv("STACKLSTM_WAIT_LIMIT_BWD_CYCLES");
    s->wait_limit_bwd = limb ? atoll(limb) : s->wait_limit;
    if ((e = allow_smem(fwd_step_tc<32>)) || (e = allow_smem(fwd_step_tc<16>)) || (e = allow_smem(fwd_step_tc<8>)) ||
        (e = allow_smem(bwd_step_tc<32>)) || (e = allow_smem(bwd_step_tc<16>)) || (e = allow_smem(dx_tc<32>)) ||
        (e = allow_smem(dx_tc<64>)) || (e = allow_smem(dx_tc<128>)) || (e = allow_smem(dx_tc<256>)))
        return e;
    if ((e = bf16_plan_dw(s))) return e;

    // persistent step kernels unless disabled (test hook, include/stacklstm.h:
    // STACKLSTM_STEP_KERNELS=1 keeps one launch per step)
    const char *per_step = getenv("STACKLSTM_STEP_KERNELS");
    if (!(per_step && atoi(per_step) != 0)) {
        if (bf16_plan_fwd_persist(s, &s->pf)) s->uf = s->pf.U;
        if (bf16_plan_bwd_persist(s, &s->pb)) s->ub = s->pb.U;
        if (bf16_plan_fwd_cluster(s, &s->fc)) {
            s->uf = s->fc.U;
            s->pf.on = 0;
        }
        bf16_plan_bwd_cluster(s, &s->bc);  // (the persistent plan stays as the fallback)
        // small batches: both directions on CUDA cores instead
        if (bf16_plan_small(s, &s->cc)) {
            s->pf.on = s->pb.on = s->fc.on = s->bc.on = 0;
            s->uf = s->ub = s->cc.U;
        }
    }
    s->sf = pick_stages(s->kcf, 4 * s->uf, ceil_div(H, s->uf) * (size_t)rt, sms);
    s->sb = pick_stages(s->kcb, s->ub, ceil_div(H, s->ub) * (size_t)rt, sms);
    s->sx = pick_stages(s->kcb, s->nx, s->nxt * ceil_div(R, kRows), sms);

    const size_t fwd_bytes = (size_t)std::max<size_t>(ceil_div(H, s->uf), s->pf.on ? s->pf.n_ct : 0) * s->kcf * 4 *
                             s->uf * 128;
    const size_t bwd_bytes = (size_t)std::max<size_t>(ceil_div(H, s->ub), s->pb.on ? s->pb.n_ct : 0) * s->kcb * s->ub *
                             128;
    const size_t dx_bytes = (size_t)s->nxt * s->kcb * s->nx * 128;
    void *p;
    if ((e = cudaMalloc(&p, fwd_bytes))) return e;
    s->allocs.push_back(p); s->w_fwd = p;
    if ((e = cudaMalloc(&p, bwd_bytes))) return e;
    s->allocs.push_back(p); s->w_bwd = p;
    if ((e = cudaMalloc(&p, dx_bytes))) return e;
    s->allocs.push_back(p); s->w_dx = p;
    if (s->fc.on) {
        if ((e = cudaMalloc(&p, bf16_fwd_cluster_block_bytes(T, B, H)))) return e;
        s->allocs.push_back(p); s->g_fcl = p;
    }
    if (s->bc.on) {
        if ((e = cudaMalloc(&p, bf16_bwd_cluster_weight_bytes(H)))) return e;
        s->allocs.push_back(p); s->w_bcl = p;
        if ((e = cudaMalloc(&p, bf16_bwd_cluster_block_bytes(T, B, H)))) return e;
        s->allocs.push_back(p); s->g_bcl = p;
    }
    if (s->cc.on) {
        if ((e = cudaMalloc(&p, bf16_small_weight_bytes(I, H, true)))) return e;
        s->allocs.push_back(p); s->w_ccf = p;
        if ((e = cudaMalloc(&p, bf16_small_weight_bytes(I, H, false)))) return e;
        s->allocs.push_back(p); s->w_ccb = p;
    }
    if ((e = cudaMalloc(&p, s->dw_part_elems * sizeof(float)))) return e;
    s->allocs.push_back(p); s->dw_part = (float *)p;
    if (s->pb.on && s->pb.KS > 1) {
        const size_t n_rt = ceil_div(B, kRows), pairs = n_rt * s->pb.n_ct;
        if ((e = cudaMalloc(&p, sizeof(float) * pairs * s->pb.KS * kRows * s->pb.U))) return e;
        s->allocs.push_back(p);
        s->split_part = (float *)p;
        if ((e = cudaMalloc(&p, sizeof(int32_t) * pairs))) return e;
        s->allocs.push_back(p);
        s->split_cnt = (int32_t *)p;
    }
    if (s->pf.on || s->pb.on) {
        if ((e = cudaMalloc(&p, 2 * sizeof(int32_t) * rt * s->cnt_stride))) return e;
        s->allocs.push_back(p);
        s->rowcnt = (int32_t *)p;
    }
    // dG is workspace: its tensor maps are fixed for the handle's lifetime
    if ((e = make_map(s->tmaps[kMapG128], s->dG, R, 4 * (uint64_t)H, kRows))) return e;
    if ((e = make_map(s->tmaps[kMapG64], s->dG, R, 4 * (uint64_t)H, kChunk))) return e;
    const uint64_t R1 = (uint64_t)(T + 1) * B;
    if ((e = make_map(s->tmaps[kMapH128], s->hr, R1, (uint64_t)H, kRows))) return e;
    if ((e = make_map(s->tmaps[kMapH64], s->hr, R1, (uint64_t)H, kChunk))) return e;
    if (s->pf.on) {
        const uint32_t ue = (uint32_t)(s->pf.U / s->pf.EP);
        if ((e = make_gates_map(s->tmaps[kMapGates], s->gates, T, B, H, ue))) return e;
        if ((e = make_hist_map(s->tmaps[kMapHistH], s->hist_h, false, T, B, H, ue))) return e;
        if ((e = make_hist_map(s->tmaps[kMapHistC], s->hist_c, true, T, B, H, ue))) return e;
    }
    return cudaSuccess;
}

cudaError_t bf16_forward_setup_x(stacklstm *s, const __nv_bfloat16 *x)
{
    const int T = s->T, B = s->B, I = s->I;
    cudaError_t e;
    if (s->push_only) {
        // the forward and the weight gradient read the inputs of the virtual steps
        if ((e = bf16_gather_push_x(s, x))) return e;
        x = (const __nv_bfloat16 *)s->x_push;
    }
    s->x_saved = x;
    if ((e = make_map(s->tmaps[kMapX128], x, (uint64_t)T * B, I, kRows))) return e;
    return make_map(s->tmaps[kMapX64], x, (uint64_t)T * B, I, kChunk);
}

cudaError_t bf16_forward_setup_state(stacklstm *s, const __nv_bfloat16 *h0, const float *c0, const __nv_bfloat16 *W)
{
    const int B = s->B, I = s->I, H = s->H;
    cudaError_t e;
    SetupArgs a{};
    a.W = W;
    a.I = I;
    a.H = H;
    // the CUDA-core kernels have weight layouts of their own
    if (s->cc.on && (e = bf16_pack_small(s, W))) return e;
    if (!s->cc.on) {
        const int nctf = std::max((int)ceil_div(H, s->uf), s->pf.on ? s->pf.n_ct : 0);
        a.wf = (__nv_bfloat16 *)s->w_fwd;
        a.uf = s->uf;
        a.kcx = s->kcx;
        a.kcf = s->kcf;
        a.n_f = (size_t)nctf * s->kcf * 4 * s->uf * kChunk;
        // the persistent and per-step backward's weight tiles (the cluster backward has its own)
        if (!s->bc.on) {
            const int nctb = std::max((int)ceil_div(H, s->ub), s->pb.on ? s->pb.n_ct : 0);
            a.wb = (__nv_bfloat16 *)s->w_bwd;
            a.ub = s->ub;
            a.n_b = (size_t)nctb * s->kcb * s->ub * kChunk;
        }
    }
    a.kcb = s->kcb;
    a.wdx = (__nv_bfloat16 *)s->w_dx;
    a.nx = s->nx;
    a.n_dx = (size_t)s->nxt * s->kcb * s->nx * kChunk;
    if (s->bc.on) {
        a.wcl = (__nv_bfloat16 *)s->w_bcl;
        a.n_ctc = s->bc.n_ct;
        a.n_cl = (size_t)s->bc.n_ct * s->bc.n_ct * 16 * 64;
    }
    a.h0 = (const uint4 *)h0;
    a.c0 = (const uint4 *)c0;
    a.hist_h = (uint4 *)s->hist_h;
    a.hr = (uint4 *)s->hr;
    a.hist_c = (uint4 *)s->hist_c;
    a.n_h = (size_t)B * H / 8;  // H % 8 == 0: whole 16-byte pieces
    a.n_c = (size_t)B * H / 4;
    // a few blocks per SM: the prepass, launched just before on the caller's stream, keeps its SMs
    const size_t n = a.n_h + a.n_c + a.n_f + a.n_b + a.n_dx + a.n_cl;
    setup_kernel<<<(unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 4)), 256, 0,
                   s->stream>>>(a);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t bf16_gather_push_x(stacklstm *s, const __nv_bfloat16 *x)
{
    const size_t rows = (size_t)s->Tr * s->B;
    const size_t n = rows * (s->I / 8);
    if (n < ((size_t)1 << 32) - (size_t)s->num_sms * 16 * 256)
        gather_push_x<uint32_t><<<grid_for(s, n), 256, 0, s->stream>>>((uint32_t)rows, (uint32_t)s->B,
                                                                        (uint32_t)(s->I / 8), s->xidx,
                                                                        (const uint4 *)x, (uint4 *)s->x_push);
    else
        gather_push_x<size_t><<<grid_for(s, n), 256, 0, s->stream>>>(rows, (size_t)s->B, (size_t)(s->I / 8), s->xidx,
                                                                      (const uint4 *)x, (uint4 *)s->x_push);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t bf16_forward_steps(stacklstm *s, const float *bias)
{
    const int T = s->Tr, B = s->B, H = s->H;
    const int nctf = std::max((int)ceil_div(H, s->uf), s->pf.on ? s->pf.n_ct : 0);
    cudaError_t e;
    if (s->cc.on) return bf16_launch_fwd_small(s, step_args(s, bias, s->w_ccf, s->kcx, s->kcf, 0));
    if (s->fc.on)
        return bf16_launch_fwd_cluster(s, step_args(s, bias, s->w_fwd, s->kcx, s->kcf, 0), map(s, kMapX64));
    if (s->pf.on)
        return bf16_launch_fwd_persist(s, step_args(s, bias, s->w_fwd, s->kcx, s->kcf, s->pf.S),
                                       map(s, B <= 64 ? kMapX64 : kMapX128), map(s, B <= 64 ? kMapH64 : kMapH128),
                                       map(s, kMapGates), map(s, kMapHistH), map(s, kMapHistC));
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

// Pointwise backward of the last step, before the reverse loop.
cudaError_t bf16_backward_setup(stacklstm *s, const float *d_top_h)
{
    StepArgs a = bwd_args(s, s->w_bwd, s->kcb, s->sb);
    a.gates_blk = s->fc.on && s->bc.on;  // the layout the cluster forward wrote for the cluster backward
    // the final top's history row of each instance (virtual, in push-only mode)
    const int32_t *ftop = (s->push_only ? s->vy : s->top) + (size_t)s->T * s->B;
    pointwise_last<<<grid_for(s, (size_t)s->B * (s->H / 8)), 256, 0, s->stream>>>(a, d_top_h, ftop);
    s->launches += 1;
    return cudaGetLastError();
}

// With dx and a plan that has spare SMs, the persistent launch also computes dx (*dx_done).
cudaError_t bf16_backward_steps(stacklstm *s, float *dx, bool *dx_done)
{
    *dx_done = false;
    const int T = s->Tr, B = s->B, H = s->H;
    cudaError_t e;
    const StepArgs a = bwd_args(s, s->w_bwd, s->kcb, s->sb);
    if (s->cc.on) return bf16_launch_bwd_small(s, bwd_args(s, s->w_ccb, s->kcb, 0));
    if (s->bc.on) return bf16_launch_bwd_cluster(s, bwd_args(s, s->w_bcl, s->kcb, 0));
    // one row tile of at most 64 instances: 64-row boxes (the rest of each stage is never
    // loaded and only feeds accumulator rows that are not stored)
    if (s->pb.on)
        return bf16_launch_bwd_persist(s, bwd_args(s, s->w_bwd, s->kcb, s->pb.S),
                                       map(s, B <= 64 ? kMapG64 : kMapG128), dx, dx_done);
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

bool bf16_can_group(stacklstm *const *hs, int n, bool fwd)
{
    for (int m = 0; m < n; ++m) {
        const stacklstm *s = hs[m];
        const PersistPlan &pl = fwd ? s->fc : s->bc;
        if (s->dt != SL_BF16 || s->cc.on || !pl.on || pl.slot != 1 || pl.n_ct != (fwd ? hs[0]->fc : hs[0]->bc).n_ct ||
            s->device != hs[0]->device)
            return false;
    }
    return true;
}

cudaError_t bf16_forward_steps_group(stacklstm *const *hs, int n, const float *const *bias, cudaStream_t st)
{
    StepArgs as[kMaxGroup];
    const CUtensorMap *tms[kMaxGroup];
    for (int m = 0; m < n; ++m) {
        as[m] = step_args(hs[m], bias[m], hs[m]->w_fwd, hs[m]->kcx, hs[m]->kcf, 0);
        tms[m] = &map(hs[m], kMapX64);
    }
    return bf16_launch_fwd_cluster_group(hs, as, tms, n, st);
}

cudaError_t bf16_backward_steps_group(stacklstm *const *hs, int n, cudaStream_t st)
{
    StepArgs as[kMaxGroup];
    for (int m = 0; m < n; ++m) as[m] = bwd_args(hs[m], hs[m]->w_bcl, hs[m]->kcb, 0);
    return bf16_launch_bwd_cluster_group(hs, as, n, st);
}

cudaError_t bf16_dx(stacklstm *s, float *dx)
{
    if (!dx) return cudaSuccess;
    const size_t R = (size_t)s->Tr * s->B;
    DxArgs d;
    d.R = R; d.I = s->I; d.KC = s->kcb; d.S = s->sx;
    d.wpack = (const uint8_t *)s->w_dx; d.dx = dx; d.limit = s->wait_limit_bwd; d.err = s->err;
    d.xidx = s->push_only ? s->xidx : nullptr;
    d.B = s->B;
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
    return bf16_launch_dw(s, map(s, kMapX64), map(s, kMapH64), map(s, kMapG64), dW, dbias);
}

// ------------------------------------------------------------ generic contraction
// D = A B^T on the tensor cores, for the parser head: A [R][K] bf16 row-major (rows lda
// elements apart, 16-byte aligned) read by TMA, B given as K-major tiles by
// bf16_pack_kmajor, D [splits][R][N] fp32 (split contraction: slab z holds the product of
// the z-th part of the K chunks; splits = 1 gives D itself).
size_t bf16_kmajor_bytes(int N, int K)
{
    const int nx = pick_dx_n(N);
    return (size_t)ceil_div(N, nx) * ceil_div(K, kChunk) * nx * 128;
}

cudaError_t bf16_pack_kmajor(const __nv_bfloat16 *src, size_t ld, bool trans, int N, int K, void *out,
                             cudaStream_t st, int num_sms)
{
    const int nx = pick_dx_n(N), KC = (int)ceil_div(K, kChunk), nt = (int)ceil_div(N, nx);
    const size_t n = (size_t)nt * KC * nx * kChunk;
    pack_kmajor<<<(unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)num_sms * 16)), 256, 0,
                  st>>>(src, ld, trans ? 1 : 0, N, K, nx, KC, nt, (__nv_bfloat16 *)out);
    return cudaGetLastError();
}

cudaError_t bf16_gemm(const __nv_bfloat16 *A, size_t lda, int R, int K, const void *bpack, int N, float *D, int splits,
                      cudaStream_t st, int num_sms, long long limit, int32_t *err)
{
    cudaError_t e;
    if ((e = get_encoder())) return e;
    alignas(64) unsigned char tm[128];
    if ((e = make_map(tm, A, (uint64_t)R, (uint64_t)K, kRows, lda))) return e;
    const int nx = pick_dx_n(N), KC = (int)ceil_div(K, kChunk), nt = (int)ceil_div(N, nx);
    splits = std::max(1, std::min(splits, KC));
    const size_t ctas = (size_t)nt * ceil_div(R, kRows) * splits;
    DxArgs d;
    d.R = (size_t)R; d.I = N; d.KC = KC;
    d.S = pick_stages(KC, nx, ctas, num_sms);
    d.wpack = (const uint8_t *)bpack; d.dx = D; d.limit = limit; d.err = err;
    d.xidx = nullptr;
    d.B = 1;
    const dim3 g(nt, ceil_div(R, kRows), splits);
    const size_t smem = smem_bytes(d.S, nx);
    const CUtensorMap &tmg = *(const CUtensorMap *)tm;
    switch (nx) {
    case 32: e = allow_smem(dx_tc<32>); if (!e) e = launch(dx_tc<32>, g, smem, st, false, tmg, d); break;
    case 64: e = allow_smem(dx_tc<64>); if (!e) e = launch(dx_tc<64>, g, smem, st, false, tmg, d); break;
    case 128: e = allow_smem(dx_tc<128>); if (!e) e = launch(dx_tc<128>, g, smem, st, false, tmg, d); break;
    default: e = allow_smem(dx_tc<256>); if (!e) e = launch(dx_tc<256>, g, smem, st, false, tmg, d); break;
    }
    return e ? e : cudaGetLastError();
}

}  // namespace sl
