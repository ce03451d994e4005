// bf16_small.cu -- the forward recurrence (Algorithm 1) and the reverse-time backward
// (Sec. 5) for small batches (B <= 32) on CUDA cores: one thread-block cluster of
// n_ct = ceil(H / 16) CTAs, each holding the weights of its 16 hidden units in shared
// memory for the whole launch. At such batch sizes a step's gate contraction (B x (I + H)
// x 4H) is too thin for the tensor cores: an M = 64 tcgen05 tile would be at least three
// quarters empty and its issue latency sets the step time, so here each step is an FFMA
// contraction (bf16 operands widened to fp32, fp32 accumulation) spread over the CTA's
// 256 threads.
//
// Per step, each CTA computes its 16 units' four gates for every row, runs the cell (or
// the pointwise backward) and stores its slice of the next step's operand (forward: the
// h_read row slice; backward: the dG row slice, 4 gates x 16 units) into every CTA of
// the cluster with distributed-shared-memory stores, then arrives on the cluster barrier
// (release); the next step waits on it (acquire) before it reads the operand. The x part
// of the forward contraction does not depend on the previous step and is computed before
// that wait. Every thread of every CTA runs the same number of barrier phases (the loops
// have no early exit), and the CTAs of a cluster are co-scheduled, so the barrier waits
// always end. Each (row, unit) has one owner thread for the whole launch: the gradient
// history needs no atomics and the backward is bitwise reproducible.
//
// The workspace is the one the tensor-core kernels use (history rows, h operand rows,
// row-major fp16 gates, bf16 dG rows), so dx and dW run unchanged after these kernels.
#include <stdio.h>

#include <algorithm>

#include "bf16_dev.cuh"

namespace sl {
namespace {

constexpr int kCcU = 16;          // hidden units per CTA
constexpr int kCcThreads = 256;   // 8 warps
constexpr int kCcWarps = kCcThreads / 32;
constexpr int kCcRedStride = 80;  // floats per reduction row: rows b, b + 1 of a warp hit distinct banks
constexpr int kCcMaxB = 32;       // rows the kernels hold (register accumulators per row)
// Largest batch the planner gives these kernels by default. Measured at I = H = 200 (one
// forward + backward pass of the parser sweep workload): B = 1, 0.597 ms here against
// 0.695 ms for the tensor-core cluster kernels (backward step 1.67 against 2.26 us, the
// forward step equal at 1.57 us); B = 8, 1.80 ms against 0.77 ms; B = 32, 6.19 against
// 0.83 ms. Per row, the FFMA contraction adds about 0.4 us a step.
constexpr int kCcCrossoverB = 1;

__device__ __forceinline__ uint32_t cc_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// address of the same shared-memory location in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t cc_mapa(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
__device__ __forceinline__ void cc_st_remote(uint32_t addr, uint4 v)
{
    asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ void cc_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cc_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

// 8 bf16 (one 16-byte piece) to fp32
__device__ __forceinline__ void unpack8_bf16(const uint4 &u, float (&v)[8])
{
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(*(const __nv_bfloat162 *)&w[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// ------------------------------------------------------------------------ forward
// Shared memory: [Ws: K x 64 bf16, row k = W row k at this CTA's 64 gate columns
// (gate-major: column g * 16 + j is gate g of unit 16 ct + j)][hbuf: 2 x BT x Hp bf16,
// h_read by step parity][xs: 2 x BT x I bf16, x by step parity][red: 8 x BT x kCcRedStride fp32]
// [hst: BT x 16 bf16, this CTA's slice of the next h_read].
__host__ __device__ constexpr size_t ccf_smem_bytes(int BT, int I, int H, int n_ct)
{
    return (size_t)(I + H) * 128 + 2u * BT * n_ct * kCcU * 2 + 2u * BT * I * 2 +
           (size_t)kCcWarps * BT * kCcRedStride * 4 + (size_t)BT * kCcU * 2;
}

struct CcArgs {
    StepArgs s;
    int n_ct;
    const __nv_bfloat16 *x;   // [T][B][I] (the forward's x, or the virtual steps' x)
    const uint8_t *wf;        // forward weight slices [n_ct][K][64] bf16
    const uint8_t *wb;        // backward weight slices [n_ct][16][4 Hp + 8] bf16
};

// acc[b][0..1] += sum over k in [k8_lo, k8_hi) x 8 of v[b][k] * W[k][2 l .. 2 l + 1], where v
// rows are `ld` bf16 apart in shared memory and W rows are 64 bf16 (this thread's two
// columns at 2 l)
template <int BT>
__device__ __forceinline__ void cc_dot(float (&acc)[BT][2], const __nv_bfloat16 *v, int ld, const __nv_bfloat16 *Ws,
                                       int k8_lo, int k8_hi, int l, int B)
{
    for (int k8 = k8_lo; k8 < k8_hi; ++k8) {
        float2 w[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            w[i] = __bfloat1622float2(*(const __nv_bfloat162 *)(Ws + (size_t)(8 * k8 + i) * 64 + 2 * l));
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= B) break;
            float xv[8];
            unpack8_bf16(*(const uint4 *)(v + (size_t)b * ld + 8 * k8), xv);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                acc[b][0] = fmaf(xv[i], w[i].x, acc[b][0]);
                acc[b][1] = fmaf(xv[i], w[i].y, acc[b][1]);
            }
        }
    }
}

template <int BT>
__global__ void __launch_bounds__(kCcThreads, 1) step_ccf(CcArgs p)
{
    const StepArgs &a = p.s;
    const int T = a.T, B = a.B, I = a.I, H = a.H, K = I + H, n_ct = p.n_ct, Hp = n_ct * kCcU;
    extern __shared__ __align__(16) uint8_t smem[];
    __nv_bfloat16 *Ws = (__nv_bfloat16 *)smem;
    __nv_bfloat16 *hbuf = Ws + (size_t)K * 64;
    __nv_bfloat16 *xs = hbuf + 2 * BT * Hp;
    float *red = (float *)(xs + 2 * BT * I);
    __nv_bfloat16 *hst = (__nv_bfloat16 *)(red + kCcWarps * BT * kCcRedStride);
    __shared__ float s_bias[4 * kCcU];
    const uint32_t ct = cc_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // weights (packed per CTA in this layout), bias, h_read(0) (every CTA reads all of it:
    // it is the initial state, no exchange needed), x of step 0
    {
        const uint4 *src = (const uint4 *)(p.wf + (size_t)ct * K * 128);
        for (int e = tid; e < K * 8; e += kCcThreads) ((uint4 *)Ws)[e] = src[e];
    }
    if (tid < 4 * kCcU) {
        const int g = tid / kCcU, u = (int)ct * kCcU + tid % kCcU;
        s_bias[tid] = u < H ? a.bias[g * H + u] : 0.0f;
    }
    for (int e = tid; e < 2 * BT * Hp; e += kCcThreads) {
        const int b = (e / Hp) % BT, k = e % Hp;
        hbuf[e] = (e < BT * Hp && b < B && k < H) ? a.hr[(size_t)b * H + k] : __float2bfloat16(0.0f);
    }
    // x of step t into xs[t & 1] by asynchronous 16-byte copies (one commit group)
    auto stage_x = [&](int t) {
        const __nv_bfloat16 *src = p.x + (size_t)t * B * I;
        const uint32_t dst = smem_u32(xs + (t & 1) * BT * I);
        for (int e = tid; e < B * I / 8; e += kCcThreads) tc::cp_async16(dst + 16u * e, src + 8 * e, 16);
        tc::cp_async_commit();
    };
    stage_x(0);
    if (T > 1) stage_x(1);

    // cell threads: unit 16 ct + j of rows tid / 16 + 16 r (RPT rows a thread)
    constexpr int RPT = (BT + 15) / 16;
    const int cj = tid % kCcU, cu = (int)ct * kCcU + cj;
    // per row: c of the state this step reads, the h of the next step's operand when that
    // is an older state, and the top indices of the next two times (loaded a step ahead, so
    // that no load waits for another)
    float c_read[RPT];
    __nv_bfloat16 hold[RPT];
    int s_nxt[RPT], s_2[RPT];
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        const int cb = tid / kCcU + 16 * r;
        c_read[r] = 0.0f;
        hold[r] = __float2bfloat16(0.0f);
        s_nxt[r] = s_2[r] = 0;
        if (cb < B && cu < H) {
            c_read[r] = a.hist_c[((size_t)a.top[cb] * B + cb) * H + cu];
            s_nxt[r] = a.top[(size_t)B + cb];
            s_2[r] = T >= 2 ? a.top[(size_t)2 * B + cb] : 0;
            if (s_nxt[r] != 1) hold[r] = a.hist_h[((size_t)s_nxt[r] * B + cb) * H + cu];
        }
    }
    // contraction ranges of this warp (8-element groups): x part, h part
    const int x8 = I / 8, h8 = H / 8;
    const int xlo = warp * x8 / kCcWarps, xhi = (warp + 1) * x8 / kCcWarps;
    const int hlo = warp * h8 / kCcWarps, hhi = (warp + 1) * h8 / kCcWarps;
    const __nv_bfloat16 *Wh = Ws + (size_t)I * 64;
    float accx[BT][2];
    if (T > 1)
        tc::cp_async_wait<1>();  // x of step 0 (x of step 1 may still be on its way)
    else
        tc::cp_async_wait<0>();
    __syncthreads();
#pragma unroll
    for (int b = 0; b < BT; ++b) accx[b][0] = accx[b][1] = 0.0f;
    cc_dot<BT>(accx, xs, I, Ws, xlo, xhi, lane, B);
    // every CTA's shared memory is initialised before any peer stores into it
    cc_arrive();
    cc_wait();

    for (int t = 0; t < T; ++t) {
        const int buf = t & 1;
        if (t > 0) cc_wait();  // h_read(t): every CTA's slice has landed in hbuf[buf]
        float acc[BT][2];
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            acc[b][0] = accx[b][0];
            acc[b][1] = accx[b][1];
        }
        cc_dot<BT>(acc, hbuf + buf * BT * Hp, Hp, Wh, hlo, hhi, lane, B);
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= B) break;
            *(float2 *)(red + (warp * BT + b) * kCcRedStride + 2 * lane) = make_float2(acc[b][0], acc[b][1]);
        }
        __syncthreads();
#pragma unroll
        for (int r = 0; r < RPT; ++r) {
            const int cb = tid / kCcU + 16 * r;
            if (cb >= B) break;
            const bool cell = cu < H;
            float z[4];
#pragma unroll
            for (int g = 0; g < 4; ++g) {
                float v = s_bias[g * kCcU + cj];
#pragma unroll
                for (int w = 0; w < kCcWarps; ++w) v += red[(w * BT + cb) * kCcRedStride + g * kCcU + cj];
                z[g] = v;
            }
            const float ig = sigm(z[0]), fg = sigm(z[1]), gg = tanh_hw(z[2]), og = sigm(z[3]);
            const float cn = fmaf(fg, c_read[r], ig * gg);
            const float hn = og * tanh_hw(cn);
            const __nv_bfloat16 hb = __float2bfloat16(hn);
            const bool is_new = s_nxt[r] == t + 1;  // step t pushed: h' is the next step's operand
            const __nv_bfloat16 hop = is_new ? hb : hold[r];
            hst[cb * kCcU + cj] = cell ? hop : __float2bfloat16(0.0f);
            if (cell) {
                // history row t + 1, the h operand row t + 1 (for the weight gradient), the gates
                const size_t w = ((size_t)(t + 1) * B + cb) * H + cu;
                a.hist_h[w] = hb;
                a.hr[w] = hop;
                a.hist_c[w] = cn;
                __half *gt = a.gates + ((size_t)t * B + cb) * 4 * H + cu;
                gt[0] = __float2half_rn(ig);
                gt[(size_t)H] = __float2half_rn(fg);
                gt[(size_t)2 * H] = __float2half_rn(gg);
                gt[(size_t)3 * H] = __float2half_rn(og);
                // the next step's operands: c of the state it reads, and (when step t + 1
                // does not push) the older state's h that is step t + 2's operand
                if (t + 1 < T) {
                    c_read[r] = is_new ? cn : a.hist_c[((size_t)s_nxt[r] * B + cb) * H + cu];
                    const int s2 = s_2[r];
                    hold[r] = s2 == t + 1 ? hb : s2 < t + 1 ? a.hist_h[((size_t)s2 * B + cb) * H + cu] : hold[r];
                    s_nxt[r] = s2;
                    s_2[r] = t + 3 <= T ? a.top[(size_t)(t + 3) * B + cb] : 0;
                }
            }
        }
        __syncthreads();
        if (t + 1 < T) {
            // this CTA's slice of h_read(t + 1) into every CTA's hbuf[buf ^ 1]
            const uint32_t dst0 = smem_u32(hbuf + (buf ^ 1) * BT * Hp + ct * kCcU);
            for (int e = tid; e < n_ct * B * 2; e += kCcThreads) {
                const int d = e / (2 * B), b = (e / 2) % B, half = e & 1;
                const uint4 v = *(const uint4 *)(hst + b * kCcU + 8 * half);
                cc_st_remote(cc_mapa(dst0 + (uint32_t)(b * Hp + 8 * half) * 2, (uint32_t)d), v);
            }
        }
        cc_arrive();
        if (t + 1 < T) {
            // the x part of step t + 1 while the other CTAs finish step t (its copies were
            // issued a step ago), then the copies of step t + 2 into the buffer step t used
            tc::cp_async_wait<0>();
            __syncthreads();
#pragma unroll
            for (int b = 0; b < BT; ++b) accx[b][0] = accx[b][1] = 0.0f;
            cc_dot<BT>(accx, xs + ((t + 1) & 1) * BT * I, I, Ws, xlo, xhi, lane, B);
            if (t + 2 < T) stage_x(t + 2);
        }
    }
    cc_wait();  // no CTA leaves while a peer may still store into its shared memory
}

// ----------------------------------------------------------------------- backward
// Shared memory: [Wt: 16 x (4 Hp + 8) bf16, row j = W row I + 16 ct + j over the gate
// columns in the order g * Hp + u (zero past H; 8 pad elements per row spread the rows'
// banks)][gbuf: 2 x BT x 4 Hp bf16, dG_t by step parity][red: 16 x BT x 16 fp32]
// [gst: BT x 64 bf16, this CTA's slice of dG_{t-1}: 4 gates x 16 units].
__host__ __device__ constexpr int ccb_row(int n_ct) { return 4 * n_ct * kCcU + 8; }
__host__ __device__ constexpr size_t ccb_smem_bytes(int BT, int n_ct)
{
    return (size_t)kCcU * ccb_row(n_ct) * 2 + 2u * BT * 4 * n_ct * kCcU * 2 + 16u * BT * kCcU * 4 +
           (size_t)BT * 4 * kCcU * 2;
}

template <int BT>
__global__ void __launch_bounds__(kCcThreads, 1) step_ccb(CcArgs p)
{
    const StepArgs &a = p.s;
    const int T = a.T, B = a.B, H = a.H, n_ct = p.n_ct, Hp = n_ct * kCcU, G4 = 4 * Hp, RS = ccb_row(n_ct);
    extern __shared__ __align__(16) uint8_t smem[];
    __nv_bfloat16 *Wt = (__nv_bfloat16 *)smem;
    __nv_bfloat16 *gbuf = Wt + kCcU * RS;
    float *red = (float *)(gbuf + 2 * BT * G4);
    __nv_bfloat16 *gst = (__nv_bfloat16 *)(red + 16 * BT * kCcU);
    const uint32_t ct = cc_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    {
        const uint4 *src = (const uint4 *)(p.wb + (size_t)ct * kCcU * RS * 2);
        for (int e = tid; e < kCcU * RS / 8; e += kCcThreads) ((uint4 *)Wt)[e] = src[e];
    }
    // dG of step T - 1 (the pointwise backward before this launch wrote it): every CTA
    // reads all of it; the other buffer starts at zero (rows >= B and units >= H stay so)
    for (int e = tid; e < 2 * BT * G4; e += kCcThreads) {
        const int b = (e / G4) % BT, c = e % G4, g = c / Hp, u = c % Hp;
        gbuf[e] = (e < BT * G4 && b < B && u < H) ? a.dG[((size_t)(T - 1) * B + b) * 4 * H + g * H + u]
                                                   : __float2bfloat16(0.0f);
    }

    // cell threads: unit 16 ct + j of rows tid / 16 + 16 r (RPT rows a thread), with the
    // operands of the step they finish next
    constexpr int RPT = (BT + 15) / 16;
    const int cj = tid % kCcU, cu = (int)ct * kCcU + cj;
    struct Ops {
        int src, s1;
        float dh_src, dh_t, dc_t, cn, cr, dc_rd, gq[4];
    };
    Ops o[RPT];
    int nsrc[RPT], ns1[RPT];  // top indices of the next step to finish (loaded a step ahead)
    auto load_ops = [&](Ops &q, int cb, int t, int src, int s1) {
        q.src = src;
        q.s1 = s1;
        q.dh_src = a.dhist_h[((size_t)q.src * B + cb) * H + cu];
        if (t >= 1) {
            const size_t wr = ((size_t)t * B + cb) * H + cu, rd = ((size_t)q.s1 * B + cb) * H + cu;
            q.dh_t = a.dhist_h[wr];
            q.dc_t = a.dhist_c[wr];
            q.cn = a.hist_c[wr];
            q.cr = a.hist_c[rd];
            q.dc_rd = a.dhist_c[rd];
            const __half *gt = a.gates + ((size_t)(t - 1) * B + cb) * 4 * H + cu;
#pragma unroll
            for (int g = 0; g < 4; ++g) q.gq[g] = __half2float(gt[(size_t)g * H]);
        }
    };
    auto top_at = [&](int t, int cb) { return t >= 0 ? a.top[(size_t)t * B + cb] : 0; };
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        o[r] = Ops{0, 0, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, {0.f, 0.f, 0.f, 0.f}};
        nsrc[r] = ns1[r] = 0;
        const int cb = tid / kCcU + 16 * r;
        if (cb < B && cu < H) {
            load_ops(o[r], cb, T - 1, top_at(T - 1, cb), top_at(T - 2, cb));
            nsrc[r] = top_at(T - 2, cb);
            ns1[r] = top_at(T - 3, cb);
        }
    }
    // contraction: lane -> unit j = lane % 16 and half lane / 16; part q = 2 warp + half
    // of the 4 Hp gate columns (Hp / 4 columns, groups of 4)
    const int uj = lane & 15, q = 2 * warp + (lane >> 4);
    const int c_lo = q * (Hp / 4), c_hi = c_lo + Hp / 4;
    __syncthreads();
    cc_arrive();
    cc_wait();

    for (int k = 0; k < T; ++k) {
        const int t = T - 1 - k, buf = k & 1;
        if (k > 0) cc_wait();  // dG_t: every CTA's slice has landed in gbuf[buf]
        float acc[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) acc[b] = 0.0f;
        const __nv_bfloat16 *gb = gbuf + buf * BT * G4;
        for (int c = c_lo; c < c_hi; c += 4) {
            const uint2 wv = *(const uint2 *)(Wt + uj * RS + c);
            const float2 w01 = __bfloat1622float2(*(const __nv_bfloat162 *)&wv.x);
            const float2 w23 = __bfloat1622float2(*(const __nv_bfloat162 *)&wv.y);
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                if (b >= B) break;
                const uint2 gv = *(const uint2 *)(gb + b * G4 + c);
                const float2 g01 = __bfloat1622float2(*(const __nv_bfloat162 *)&gv.x);
                const float2 g23 = __bfloat1622float2(*(const __nv_bfloat162 *)&gv.y);
                acc[b] = fmaf(g01.x, w01.x, acc[b]);
                acc[b] = fmaf(g01.y, w01.y, acc[b]);
                acc[b] = fmaf(g23.x, w23.x, acc[b]);
                acc[b] = fmaf(g23.y, w23.y, acc[b]);
            }
        }
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (b >= B) break;
            red[(q * BT + b) * kCcU + uj] = acc[b];
        }
        __syncthreads();
#pragma unroll
        for (int r = 0; r < RPT; ++r) {
            const int cb = tid / kCcU + 16 * r;
            if (cb >= B) break;
            const bool cell = cu < H;
            const Ops &q = o[r];
            float dr = 0.0f;  // dh_read of this row and unit: the 16 parts in part order
#pragma unroll
            for (int i = 0; i < 16; ++i) dr += red[(i * BT + cb) * kCcU + cj];
            const float v = q.dh_src + dr;
            if (t >= 1) {
                // the pointwise backward of step t - 1 (the state it wrote is row t)
                const float dh = q.src == t ? v : q.dh_t;
                const float tcn = tanh_hw(q.cn);
                const float dc = q.dc_t + dh * q.gq[3] * (1.0f - tcn * tcn);
                float d[4];
                d[0] = dc * q.gq[2] * q.gq[0] * (1.0f - q.gq[0]);
                d[1] = dc * q.cr * q.gq[1] * (1.0f - q.gq[1]);
                d[2] = dc * q.gq[0] * (1.0f - q.gq[2] * q.gq[2]);
                d[3] = dh * tcn * q.gq[3] * (1.0f - q.gq[3]);
                const float dcr = q.dc_rd + dc * q.gq[1];
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const __nv_bfloat16 dg = __float2bfloat16(d[g]);
                    gst[cb * 4 * kCcU + g * kCcU + cj] = cell ? dg : __float2bfloat16(0.0f);
                    if (cell) a.dG[((size_t)(t - 1) * B + cb) * 4 * H + g * H + cu] = dg;
                }
                if (cell) a.dhist_c[((size_t)q.s1 * B + cb) * H + cu] = dcr;
            }
            if (cell) a.dhist_h[((size_t)q.src * B + cb) * H + cu] = v;
        }
        __syncthreads();
        if (t >= 1) {
            // this CTA's slice of dG_{t-1} into every CTA's gbuf[buf ^ 1]
            const uint32_t dst0 = smem_u32(gbuf + (buf ^ 1) * BT * G4 + ct * kCcU);
            for (int e = tid; e < n_ct * B * 8; e += kCcThreads) {
                const int d = e / (8 * B), b = (e / 8) % B, g = (e / 2) & 3, half = e & 1;
                const uint4 v = *(const uint4 *)(gst + b * 4 * kCcU + g * kCcU + 8 * half);
                cc_st_remote(cc_mapa(dst0 + (uint32_t)(b * G4 + g * Hp + 8 * half) * 2, (uint32_t)d), v);
            }
        }
        cc_arrive();
        if (t >= 1)  // after this thread's own stores above
#pragma unroll
            for (int r = 0; r < RPT; ++r) {
                const int cb = tid / kCcU + 16 * r;
                if (cb < B && cu < H) {
                    load_ops(o[r], cb, t - 1, nsrc[r], ns1[r]);
                    nsrc[r] = top_at(t - 2, cb);
                    ns1[r] = top_at(t - 3, cb);
                }
            }
    }
    cc_wait();  // no CTA leaves while a peer may still store into its shared memory
}

// --------------------------------------------------------------------- packing
// Forward slices [n_ct][K][64]: row k of CTA ct is W row k at gate column g * H + 16 ct + j
// for column g * 16 + j (zero past H).
__global__ void pack_ccf(const __nv_bfloat16 *__restrict__ W, int K, int H, int n_ct, __nv_bfloat16 *__restrict__ out)
{
    const size_t n = (size_t)n_ct * K * 64;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int c = (int)(e % 64);
        const size_t rk = e / 64;
        const int k = (int)(rk % K), ct = (int)(rk / K);
        const int u = ct * kCcU + c % kCcU, g = c / kCcU;
        out[e] = u < H ? W[(size_t)k * 4 * H + g * H + u] : __float2bfloat16(0.0f);
    }
}

// Backward slices [n_ct][16][4 Hp + 8]: row j of CTA ct is W row I + 16 ct + j at gate
// column g * H + u for position g * Hp + u (zero past H and in the pad).
__global__ void pack_ccb(const __nv_bfloat16 *__restrict__ W, int I, int H, int n_ct, __nv_bfloat16 *__restrict__ out)
{
    const int Hp = n_ct * kCcU, RS = ccb_row(n_ct);
    const size_t n = (size_t)n_ct * kCcU * RS;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int c = (int)(e % RS);
        const size_t rj = e / RS;
        const int j = (int)(rj % kCcU), ct = (int)(rj / kCcU);
        const int unit = ct * kCcU + j, g = c / Hp, u = c % Hp;
        out[e] = (c < 4 * Hp && unit < H && u < H) ? W[(size_t)(I + unit) * 4 * H + g * H + u]
                                                   : __float2bfloat16(0.0f);
    }
}

int cc_tier(int B) { return B <= 1 ? 1 : B <= 2 ? 2 : B <= 4 ? 4 : B <= 8 ? 8 : B <= 16 ? 16 : 32; }

template <int BT>
const void *ccf_fn() { return (const void *)step_ccf<BT>; }
template <int BT>
const void *ccb_fn() { return (const void *)step_ccb<BT>; }
const void *cc_fn(bool fwd, int BT)
{
    switch (BT) {
    case 1: return fwd ? ccf_fn<1>() : ccb_fn<1>();
    case 2: return fwd ? ccf_fn<2>() : ccb_fn<2>();
    case 4: return fwd ? ccf_fn<4>() : ccb_fn<4>();
    case 8: return fwd ? ccf_fn<8>() : ccb_fn<8>();
    case 16: return fwd ? ccf_fn<16>() : ccb_fn<16>();
    default: return fwd ? ccf_fn<32>() : ccb_fn<32>();
    }
}

// one cluster of n_ct CTAs for all T steps
cudaError_t cc_launch(stacklstm *s, bool fwd, const CcArgs &p, size_t smem)
{
    const void *fn = cc_fn(fwd, cc_tier(s->B));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(p.n_ct);
    cfg.blockDim = dim3(kCcThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s->stream;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = p.n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    void *argv[] = {(void *)&p};
    cudaError_t e = cudaLaunchKernelExC(&cfg, fn, argv);
    if (e) return e;
    s->launches += 1;
    return cudaGetLastError();
}

}  // namespace

// Batches up to kCcMaxB: the CUDA-core cluster kernels when the shape fits (at most 16
// CTAs of 16 units; both footprints within shared memory; the cluster co-resident) and
// B is at most the crossover below which they beat the tensor-core cluster kernels
// (measured on this GPU at I = H = 200). Test hook (include/stacklstm.h):
// STACKLSTM_CUDA_CORE=0 never, =1 whenever the shape fits.
bool bf16_plan_small(stacklstm *s, PersistPlan *pl)
{
    pl->on = 0;
    const char *env = getenv("STACKLSTM_CUDA_CORE");
    const int want = env ? atoi(env) : -1;
    if (want == 0) return false;
    const int n_ct = (int)ceil_div(s->H, kCcU), BT = cc_tier(s->B);
    if (s->B > kCcMaxB || n_ct > 16 || s->I % 8 || s->H % 8) return false;
    if (want < 0 && s->B > kCcCrossoverB) return false;
    const size_t sf = ccf_smem_bytes(BT, s->I, s->H, n_ct), sb = ccb_smem_bytes(BT, n_ct);
    if (sf > kSmemCap || sb > kSmemCap) return false;
    for (int dir = 0; dir < 2; ++dir) {
        const void *fn = cc_fn(dir == 0, BT);
        const size_t smem = dir == 0 ? sf : sb;
        if (smem_at_least(fn, smem) != cudaSuccess ||
            (n_ct > 8 && cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)) {
            cudaGetLastError();
            return false;
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(n_ct);
        cfg.blockDim = dim3(kCcThreads);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = n_ct;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int clusters = 0;
        if (cudaOccupancyMaxActiveClusters(&clusters, fn, &cfg) != cudaSuccess || clusters < 1) {
            cudaGetLastError();
            return false;
        }
    }
    pl->on = 1;
    pl->U = kCcU;
    pl->EP = 1;
    pl->n_ct = n_ct;
    pl->cl = n_ct;
    pl->slot = 1;
    pl->smem = (unsigned)sf;
    pl->threads = kCcThreads;
    return true;
}

size_t bf16_small_weight_bytes(int I, int H, bool fwd)
{
    const size_t n_ct = ceil_div(H, kCcU);
    return fwd ? n_ct * (size_t)(I + H) * 64 * 2 : n_ct * kCcU * (size_t)ccb_row((int)n_ct) * 2;
}

cudaError_t bf16_pack_small(stacklstm *s, const __nv_bfloat16 *W)
{
    const int n_ct = s->cc.n_ct;
    const size_t nf = (size_t)n_ct * (s->I + s->H) * 64, nb = (size_t)n_ct * kCcU * ccb_row(n_ct);
    pack_ccf<<<(unsigned)std::min<size_t>(ceil_div(nf, 256), 4096), 256, 0, s->stream>>>(
        W, s->I + s->H, s->H, n_ct, (__nv_bfloat16 *)s->w_ccf);
    pack_ccb<<<(unsigned)std::min<size_t>(ceil_div(nb, 256), 4096), 256, 0, s->stream>>>(
        W, s->I, s->H, n_ct, (__nv_bfloat16 *)s->w_ccb);
    s->launches += 2;
    return cudaGetLastError();
}

cudaError_t bf16_launch_fwd_small(stacklstm *s, const StepArgs &a)
{
    CcArgs p{};
    p.s = a;
    p.s.gates_blk = 0;
    p.n_ct = s->cc.n_ct;
    p.x = (const __nv_bfloat16 *)s->x_saved;
    p.wf = (const uint8_t *)s->w_ccf;
    p.wb = (const uint8_t *)s->w_ccb;
    return cc_launch(s, true, p, ccf_smem_bytes(cc_tier(s->B), s->I, s->H, p.n_ct));
}

cudaError_t bf16_launch_bwd_small(stacklstm *s, const StepArgs &a)
{
    CcArgs p{};
    p.s = a;
    p.s.gates_blk = 0;
    p.n_ct = s->cc.n_ct;
    p.x = (const __nv_bfloat16 *)s->x_saved;
    p.wf = (const uint8_t *)s->w_ccf;
    p.wb = (const uint8_t *)s->w_ccb;
    return cc_launch(s, false, p, ccb_smem_bytes(cc_tier(s->B), p.n_ct));
}

}  // namespace sl
