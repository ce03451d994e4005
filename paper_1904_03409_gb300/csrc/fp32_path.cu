// fp32_path.cu -- the fp32 homogenized StackLSTM step on CUDA cores (no tensor cores,
// no TF32). It serves small problems, where B * 4H is too small for a dense tensor-core
// contraction, and is the full-precision counterpart of the bf16 path. With B * H <= 1024
// each direction runs all its steps in one CTA (fwd_seq_f32, bwd_seq_f32); otherwise:
//
// Forward, one launch per step t (Algorithm 1): every instance reads history row
// top[t] (the state at its stack top), computes z = [x_t ; h_read] W + bias, applies the
// LSTM cell and writes history row t + 1 (its slot p_t + 1). No step branches on an op.
// Backward, two launches per step in reverse time (Sec. 5): the pointwise kernel turns
// (dh', dc') of row t + 1 into gate gradients dG_t and adds dc_read to row top[t]; the
// contraction kernel adds dh_read = dG_t W_h^T to row top[t]. Each (row, column) of the
// gradient history has exactly one writer per launch, so no atomics are needed and the
// summation order is fixed. dx = dG W_x^T, dW = [x ; h_read]^T dG and dbias = sum dG are
// taken after the loop in a fixed order.
#include <stdlib.h>

#include <algorithm>
#include <string>

#include "common.cuh"

namespace sl {
namespace {

__device__ __forceinline__ float sigmoidf(float z) { return 1.0f / (1.0f + expf(-z)); }

// grid (ceil(H / blockDim.x), B); one thread per hidden unit j of instance b.
__global__ void fwd_step_f32(int t, int B, int I, int H, const float *__restrict__ x,
                             const float *__restrict__ W, const float *__restrict__ bias,
                             const int32_t *__restrict__ top, float *__restrict__ hist_h,
                             float *__restrict__ hist_c, float *__restrict__ gates,
                             float *__restrict__ a_rm)
{
    extern __shared__ float a_s[];  // [I + H]: the contraction operand [x_t ; h_read]
    const int b = blockIdx.y, K = I + H, G = 4 * H;
    const int src = top[(size_t)t * B + b];
    const float *xt = x + ((size_t)t * B + b) * I;
    const float *hr = hist_h + ((size_t)src * B + b) * H;
    for (int k = threadIdx.x; k < K; k += blockDim.x) a_s[k] = k < I ? xt[k] : hr[k - I];
    __syncthreads();
    if (blockIdx.x == 0)
        for (int k = threadIdx.x; k < K; k += blockDim.x) a_rm[((size_t)t * B + b) * K + k] = a_s[k];
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= H) return;
    float zi = bias[j], zf = bias[H + j], zg = bias[2 * H + j], zo = bias[3 * H + j];
    for (int k = 0; k < K; ++k) {
        const float a = a_s[k];
        const float *Wk = W + (size_t)k * G;
        zi = fmaf(a, Wk[j], zi);
        zf = fmaf(a, Wk[H + j], zf);
        zg = fmaf(a, Wk[2 * H + j], zg);
        zo = fmaf(a, Wk[3 * H + j], zo);
    }
    const float ig = sigmoidf(zi), fg = sigmoidf(zf), gg = tanhf(zg), og = sigmoidf(zo);
    const float cr = hist_c[((size_t)src * B + b) * H + j];
    const float cn = fmaf(fg, cr, ig * gg);
    const float hn = og * tanhf(cn);
    const size_t w = ((size_t)(t + 1) * B + b) * H + j;
    hist_h[w] = hn;
    hist_c[w] = cn;
    float *gt = gates + ((size_t)t * B + b) * G;
    gt[j] = ig;
    gt[H + j] = fg;
    gt[2 * H + j] = gg;
    gt[3 * H + j] = og;
}

// The forward setup in one launch: history row 0 = (h0, c0), the initial state (stack
// slot 0), and W^T (out[c][r] = in[r][c], R x C) for the backward contractions, so that the
// backward needs nothing the caller owns.
__global__ void setup_f32(int n0, const float *__restrict__ h0, const float *__restrict__ c0,
                          float *__restrict__ hist_h, float *__restrict__ hist_c, int R, int C,
                          const float *__restrict__ in, float *__restrict__ out)
{
    const size_t n = (size_t)R * C, stride = (size_t)gridDim.x * blockDim.x;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n + n0; e += stride) {
        if (e < (size_t)n0) {
            hist_h[e] = h0[e];
            hist_c[e] = c0[e];
        } else {
            const size_t f = e - n0, r = f / C, c = f - r * C;
            out[c * R + r] = in[f];
        }
    }
}

// Pointwise backward of step t; one thread per (b, j).
__global__ void bwd_pointwise_f32(int t, int B, int H, const int32_t *__restrict__ top,
                                  const float *__restrict__ gates, const float *__restrict__ hist_c,
                                  const float *__restrict__ dhist_h, float *__restrict__ dhist_c,
                                  float *__restrict__ dG)
{
    const size_t n = (size_t)B * H;
    const int G = 4 * H;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int b = (int)(e / H), j = (int)(e - (size_t)b * H);
        const int src = top[(size_t)t * B + b];
        const size_t wr = ((size_t)(t + 1) * B + b) * H + j;  // the state step t wrote
        const size_t rd = ((size_t)src * B + b) * H + j;      // the state step t read
        const float dh = dhist_h[wr], dcn = dhist_c[wr];
        const float *gt = gates + ((size_t)t * B + b) * G;
        const float ig = gt[j], fg = gt[H + j], gg = gt[2 * H + j], og = gt[3 * H + j];
        const float tc = tanhf(hist_c[wr]);
        const float dc = dcn + dh * og * (1.0f - tc * tc);
        float *dg = dG + ((size_t)t * B + b) * G;
        dg[j] = dc * gg * ig * (1.0f - ig);
        dg[H + j] = dc * hist_c[rd] * fg * (1.0f - fg);
        dg[2 * H + j] = dc * ig * (1.0f - gg * gg);
        dg[3 * H + j] = dh * tc * og * (1.0f - og);
        dhist_c[rd] += dc * fg;
    }
}

// dh_read = dG_t W_h^T added to row top[t]; grid (ceil(H / blockDim.x), B). P (1, 2 or 4,
// from the shape: fwd_seq_threads_per_unit) is the one-CTA backward's split of the 4H sum.
__global__ void bwd_contract_f32(int t, int B, int I, int H, int P, const int32_t *__restrict__ top,
                                 const float *__restrict__ WT, const float *__restrict__ dG,
                                 float *__restrict__ dhist_h)
{
    extern __shared__ float g_s[];  // [4H]
    const int b = blockIdx.y, G = 4 * H, K = I + H;
    const float *dg = dG + ((size_t)t * B + b) * G;
    for (int n = threadIdx.x; n < G; n += blockDim.x) g_s[n] = dg[n];
    __syncthreads();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= H) return;
    // P partial sums over consecutive quarters (halves, the whole) of the 4H gate columns,
    // added in part order: the one-CTA backward's split, in one thread
    float acc = 0.0f;
    for (int p = 0; p < P; ++p) {
        float sp = 0.0f;
        for (int n = p * (G / P); n < (p + 1) * (G / P); ++n) sp = fmaf(g_s[n], WT[(size_t)n * K + I + k], sp);
        acc = p == 0 ? sp : acc + sp;
    }
    const int src = top[(size_t)t * B + b];
    dhist_h[((size_t)src * B + b) * H + k] += acc;
}

// dx[r] = dG[r] W_x^T for every row r = t * B + b; grid (ceil(I / blockDim.x), T * B).
__global__ void dx_f32(int I, int H, const float *__restrict__ WT, const float *__restrict__ dG,
                       float *__restrict__ dx)
{
    extern __shared__ float g_s[];
    const size_t r = blockIdx.y;
    const int G = 4 * H, K = I + H;
    for (int n = threadIdx.x; n < G; n += blockDim.x) g_s[n] = dG[r * G + n];
    __syncthreads();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= I) return;
    float acc = 0.0f;
    for (int n0 = 0; n0 < G; n0 += 8) {  // eight weights loaded, then used in order
        float wv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) wv[i] = n0 + i < G ? WT[(size_t)(n0 + i) * K + k] : 0.0f;
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (n0 + i < G) acc = fmaf(g_s[n0 + i], wv[i], acc);
    }
    dx[r * I + k] = acc;
}

// dW[k][n] = sum_r a_rm[r][k] dG[r][n] and dbias[n] = sum_r dG[r][n], r ascending, with
// compensated (Kahan) summation so long fp32 sums keep their accuracy.
__global__ void dw_f32(size_t R, int K, int G, const float *__restrict__ a_rm, const float *__restrict__ dG,
                       float *__restrict__ dW, float *__restrict__ dbias)
{
    const size_t n_out = (size_t)(K + 1) * G;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n_out; e += (size_t)gridDim.x * blockDim.x) {
        const int k = (int)(e / G), n = (int)(e - (size_t)k * G);
        float acc = 0.0f, comp = 0.0f;
        // eight rows' operands loaded before they are summed (in row order), so that their
        // loads are in flight together
        for (size_t r0 = 0; r0 < R; r0 += 8) {
            float av[8], gv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const size_t r = r0 + i;
                av[i] = r < R && k < K ? a_rm[r * K + k] : 1.0f;
                gv[i] = r < R ? dG[r * G + n] : 0.0f;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (r0 + i < R) {
                    const float term = av[i] * gv[i];
                    const float y = term - comp;
                    const float t = acc + y;
                    comp = (t - acc) - y;
                    acc = t;
                }
        }
        if (k < K) {
            if (dW) dW[(size_t)k * G + n] = acc;
        } else if (dbias) {
            dbias[n] = acc;
        }
    }
}

// Small problems (B * H <= 1024, and the whole history in shared memory): all T steps of a
// direction in one CTA, P threads per (instance b, unit j) (as many of 4, 2, 1 as 1024 threads
// allow), __syncthreads() between the phases of a step instead of a launch per step, and
// every row a step reads taken from shared memory (the rows go to global memory as they are
// written). The forward's P threads of a unit split its four gates' dot products, the
// backward's its 4H-long contraction (in P consecutive parts, added in part order). The
// arithmetic of each element is that of the per-step kernels above (the same operands, k and
// n ascending with fmaf, the same P parts), so both give the same bits.
// Shared memory: forward [B][K] operands, [K][4H] W, [T+1][B][H] h and c, [T][B][I] x,
// [T+1][B] tops;
// backward [4H][H] W_h^T, [T+1][B][H] c, dh and dc, [B][4H] the step's dG, [T+1][B] tops.
size_t fwd_seq_smem(int T, int B, int I, int H)
{
    const size_t K = (size_t)I + H, G = 4 * (size_t)H, R = (size_t)(T + 1) * B;
    return sizeof(float) * ((size_t)B * K + K * G + 2 * R * H + (size_t)T * B * I) + sizeof(int32_t) * R;
}
size_t bwd_seq_smem(int T, int B, int H)
{
    const size_t G = 4 * (size_t)H, R = (size_t)(T + 1) * B;
    return sizeof(float) * (G * H + 3 * R * H + (size_t)B * G) + sizeof(int32_t) * R;
}
// threads per (instance, unit) of the one-CTA forward: as many of 4, 2, 1 as 1024 allow
int fwd_seq_threads_per_unit(int B, int H) { return B * H * 4 <= 1024 ? 4 : B * H * 2 <= 1024 ? 2 : 1; }

// P threads per (instance, unit), P in {1, 2, 4}: each runs the dot products of 4 / P of the
// unit's gates (every gate's fmaf chain as in fwd_step_f32, so the results are the same bit for
// bit), and the first of them collects the four by shuffles for the cell.
__global__ void __launch_bounds__(1024) fwd_seq_f32(int T, int B, int I, int H, int P, const float *__restrict__ x,
                                                    const float *__restrict__ W, const float *__restrict__ bias,
                                                    const int32_t *__restrict__ top, float *__restrict__ hist_h,
                                                    float *__restrict__ hist_c, float *__restrict__ gates,
                                                    float *__restrict__ a_rm)
{
    extern __shared__ float sm[];
    const int K = I + H, G = 4 * H, tid = threadIdx.x, u = tid / P, part = tid - u * P, GP = 4 / P;
    const int b = u / H, j = u - b * H;
    const bool mine = u < B * H;
    const int lane = tid & 31;
    const size_t R = (size_t)(T + 1) * B;
    float *a_s = sm, *w_s = a_s + (size_t)B * K, *h_s = w_s + (size_t)K * G, *c_s = h_s + R * H;
    float *x_s = c_s + R * H;
    int32_t *top_s = (int32_t *)(x_s + (size_t)T * B * I);
    for (size_t e = tid; e < (size_t)K * G; e += blockDim.x) w_s[e] = W[e];
    for (size_t e = tid; e < (size_t)T * B * I; e += blockDim.x) x_s[e] = x[e];
    for (size_t e = tid; e < R; e += blockDim.x) top_s[e] = top[e];
    for (int e = tid; e < B * H; e += blockDim.x) {  // row 0: the initial state
        h_s[e] = hist_h[e];
        c_s[e] = hist_c[e];
    }
    __syncthreads();
    for (int t = 0; t < T; ++t) {
        for (int e = tid; e < B * K; e += blockDim.x) {
            const int bb = e / K, k = e - bb * K;
            const int src = top_s[t * B + bb];
            const float v = k < I ? x_s[((size_t)t * B + bb) * I + k] : h_s[((size_t)src * B + bb) * H + (k - I)];
            a_s[e] = v;
            a_rm[((size_t)t * B + bb) * K + k] = v;
        }
        __syncthreads();
        float z[4] = {0.f, 0.f, 0.f, 0.f};  // gates part * GP .. + GP - 1 of unit (b, j)
        if (mine) {
            const float *as = a_s + (size_t)b * K;
#pragma unroll
            for (int i = 0; i < 4; ++i)
                if (i < GP) {
                    const int gc = (part * GP + i) * H + j;
                    float zz = bias[gc];
                    for (int k = 0; k < K; ++k) zz = fmaf(as[k], w_s[(size_t)k * G + gc], zz);
                    z[i] = zz;
                }
        }
        // gate g of the unit is value g mod GP of its part g / GP: to the unit's first thread
        float zg4[4];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            float v = z[0];
#pragma unroll
            for (int i = 1; i < 4; ++i)
                if (g % GP == i) v = z[i];
            zg4[g] = __shfl_sync(0xffffffffu, v, (lane & ~(P - 1)) + g / GP);
        }
        if (mine && part == 0) {
            const float zi = zg4[0], zf = zg4[1], zg = zg4[2], zo = zg4[3];
            const float ig = sigmoidf(zi), fg = sigmoidf(zf), gg = tanhf(zg), og = sigmoidf(zo);
            const int src = top_s[t * B + b];
            const float cr = c_s[((size_t)src * B + b) * H + j];
            const float cn = fmaf(fg, cr, ig * gg);
            const float hn = og * tanhf(cn);
            const size_t w = ((size_t)(t + 1) * B + b) * H + j;
            h_s[w] = hn;
            c_s[w] = cn;
            hist_h[w] = hn;
            hist_c[w] = cn;
            float *gt = gates + ((size_t)t * B + b) * G;
            gt[j] = ig;
            gt[H + j] = fg;
            gt[2 * H + j] = gg;
            gt[3 * H + j] = og;
        }
        __syncthreads();  // row t + 1 is complete before a later step reads it
    }
}

__global__ void __launch_bounds__(1024) bwd_seq_f32(int T, int B, int I, int H, int P, const int32_t *__restrict__ top,
                                                    const float *__restrict__ gates, const float *__restrict__ hist_c,
                                                    const float *__restrict__ WT, float *__restrict__ dhist_h,
                                                    float *__restrict__ dhist_c, float *__restrict__ dG)
{
    extern __shared__ float sm[];
    // P threads per (instance, unit): the unit's first runs the pointwise backward; all P the
    // contraction, part p over gate columns [p G / P, (p + 1) G / P), summed in part order
    const int K = I + H, G = 4 * H, tid = threadIdx.x, u = tid / P, part = tid - u * P;
    const int b = u / H, j = u - b * H, lane = tid & 31;
    const bool unit = u < B * H, mine = unit && part == 0;
    const size_t R = (size_t)(T + 1) * B;
    float *wh_s = sm, *c_s = wh_s + (size_t)G * H, *dh_s = c_s + R * H, *dc_s = dh_s + R * H;
    float *dg_s = dc_s + R * H;  // [B][4H]: dG of the current step
    int32_t *top_s = (int32_t *)(dg_s + (size_t)B * G);
    for (int e = tid; e < G * H; e += blockDim.x) wh_s[e] = WT[(size_t)(e / H) * K + I + e % H];
    for (size_t e = tid; e < R * H; e += blockDim.x) {
        c_s[e] = hist_c[e];
        dh_s[e] = dhist_h[e];  // the seeded loss gradients (zero elsewhere)
        dc_s[e] = dhist_c[e];
    }
    for (size_t e = tid; e < R; e += blockDim.x) top_s[e] = top[e];
    // this thread's four activated gates of the next step processed (loaded a step ahead)
    float gn[4] = {0.f, 0.f, 0.f, 0.f};
    if (mine && T >= 1)
        for (int g = 0; g < 4; ++g) gn[g] = gates[((size_t)(T - 1) * B + b) * G + g * H + j];
    __syncthreads();
    for (int t = T - 1; t >= 0; --t) {
        const int src = unit ? top_s[t * B + b] : 0;
        if (mine) {
            // pointwise backward of step t (bwd_pointwise_f32)
            const float ig = gn[0], fg = gn[1], gg = gn[2], og = gn[3];
            if (t >= 1)
                for (int g = 0; g < 4; ++g) gn[g] = gates[((size_t)(t - 1) * B + b) * G + g * H + j];
            const size_t wr = ((size_t)(t + 1) * B + b) * H + j, rd = ((size_t)src * B + b) * H + j;
            const float dh = dh_s[wr], dcn = dc_s[wr];
            const float tc = tanhf(c_s[wr]);
            const float dc = dcn + dh * og * (1.0f - tc * tc);
            float *dg = dg_s + (size_t)b * G;
            float *dgo = dG + ((size_t)t * B + b) * G;
            dgo[j] = dg[j] = dc * gg * ig * (1.0f - ig);
            dgo[H + j] = dg[H + j] = dc * c_s[rd] * fg * (1.0f - fg);
            dgo[2 * H + j] = dg[2 * H + j] = dc * ig * (1.0f - gg * gg);
            dgo[3 * H + j] = dg[3 * H + j] = dh * tc * og * (1.0f - og);
            dc_s[rd] += dc * fg;
        }
        __syncthreads();  // dG_t complete
        // dh_read = dG_t W_h^T added to the row step t read (bwd_contract_f32)
        float sp = 0.0f;
        if (unit) {
            const float *dg = dg_s + (size_t)b * G;
            for (int n = part * (G / P); n < (part + 1) * (G / P); ++n) sp = fmaf(dg[n], wh_s[n * H + j], sp);
        }
        float acc = sp;
        for (int p = 1; p < P; ++p) acc = acc + __shfl_sync(0xffffffffu, sp, (lane & ~(P - 1)) + p);
        if (mine) dh_s[((size_t)src * B + b) * H + j] += acc;
        __syncthreads();  // the row's gradient is complete before step t - 1 reads it
    }
    // out: the gradient history (rows 0..T: dh0, dc0 among them)
    for (size_t e = tid; e < R * H; e += blockDim.x) {
        dhist_h[e] = dh_s[e];
        dhist_c[e] = dc_s[e];
    }
}

unsigned grid_for(const stacklstm *s, size_t n, int threads)
{
    return (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, threads), (size_t)s->num_sms * 32));
}

}  // namespace

std::string fp32_describe(stacklstm *s)
{
    // test hook (include/stacklstm.h): STACKLSTM_STEP_KERNELS=1 keeps one launch per step
    const char *per_step = getenv("STACKLSTM_STEP_KERNELS");
    int optin = 0;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, s->device) != cudaSuccess) {
        cudaGetLastError();
        optin = 48 * 1024;
    }
    const size_t cap = (size_t)optin - 1024;
    s->fp32_one_cta = s->B * s->H <= 1024 && fwd_seq_smem(s->T, s->B, s->I, s->H) <= cap &&
                      bwd_seq_smem(s->T, s->B, s->H) <= cap && !(per_step && atoi(per_step) != 0);
    if (s->fp32_one_cta && (smem_at_least((const void *)fwd_seq_f32, fwd_seq_smem(s->T, s->B, s->I, s->H)) ||
                            smem_at_least((const void *)bwd_seq_f32, bwd_seq_smem(s->T, s->B, s->H)))) {
        cudaGetLastError();
        s->fp32_one_cta = 0;
    }
    return s->fp32_one_cta ? "fp32 CUDA cores; every step of each direction in one CTA"
                           : "fp32 CUDA cores; one launch per step";
}

cudaError_t fp32_forward_setup(stacklstm *s, const float *h0, const float *c0, const float *W)
{
    const int B = s->B, I = s->I, H = s->H, K = I + H, G = 4 * H;
    setup_f32<<<grid_for(s, (size_t)K * G + (size_t)B * H, 256), 256, 0, s->stream>>>(
        B * H, h0, c0, (float *)s->hist_h, s->hist_c, K, G, W, (float *)s->w_fwd);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t fp32_forward_steps(stacklstm *s, const float *x, const float *W, const float *bias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H, K = I + H;
    if (s->fp32_one_cta) {
        (void)K;
        const int P = fwd_seq_threads_per_unit(B, H);
        fwd_seq_f32<<<1, (unsigned)ceil_div(B * H * P, 32) * 32, fwd_seq_smem(T, B, I, H), s->stream>>>(
            T, B, I, H, P, x, W, bias, s->top, (float *)s->hist_h, s->hist_c, (float *)s->gates, (float *)s->a_rm);
        s->launches += 1;
        return cudaGetLastError();
    }
    const int threads = std::min(128, ((H + 31) / 32) * 32);
    const dim3 grid(ceil_div(H, threads), B);
    const size_t smem = sizeof(float) * K;
    for (int t = 0; t < T; ++t)
        fwd_step_f32<<<grid, threads, smem, s->stream>>>(t, B, I, H, x, W, bias, s->top, (float *)s->hist_h,
                                                          s->hist_c, (float *)s->gates, (float *)s->a_rm);
    s->launches += T;
    return cudaGetLastError();
}

cudaError_t fp32_backward_steps(stacklstm *s)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H, G = 4 * H;
    const float *WT = (const float *)s->w_fwd;
    float *dG = (float *)s->dG;
    if (s->fp32_one_cta) {
        const int P = fwd_seq_threads_per_unit(B, H);
        bwd_seq_f32<<<1, (unsigned)ceil_div(B * H * P, 32) * 32, bwd_seq_smem(T, B, H), s->stream>>>(
            T, B, I, H, P, s->top, (const float *)s->gates, s->hist_c, WT, s->dhist_h, s->dhist_c, dG);
        s->launches += 1;
        return cudaGetLastError();
    }
    const int threads = std::min(128, ((H + 31) / 32) * 32);
    const unsigned pw_grid = grid_for(s, (size_t)B * H, 256);
    for (int t = T - 1; t >= 0; --t) {
        bwd_pointwise_f32<<<pw_grid, 256, 0, s->stream>>>(t, B, H, s->top, (const float *)s->gates, s->hist_c,
                                                          s->dhist_h, s->dhist_c, dG);
        bwd_contract_f32<<<dim3(ceil_div(H, threads), B), threads, sizeof(float) * G, s->stream>>>(
            t, B, I, H, fwd_seq_threads_per_unit(B, H), s->top, WT, dG, s->dhist_h);
    }
    s->launches += 2 * T;
    return cudaGetLastError();
}

cudaError_t fp32_dx(stacklstm *s, float *dx)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H, G = 4 * H;
    const float *WT = (const float *)s->w_fwd;
    const float *dG = (const float *)s->dG;
    if (dx && T > 0) {
        const int tx = std::min(128, ((I + 31) / 32) * 32);
        // grid.y is limited to 65535 rows per launch
        for (size_t r0 = 0; r0 < (size_t)T * B; r0 += 65535) {
            const unsigned rows = (unsigned)std::min<size_t>(65535, (size_t)T * B - r0);
            dx_f32<<<dim3(ceil_div(I, tx), rows), tx, sizeof(float) * G, s->stream>>>(I, H, WT, dG + r0 * G,
                                                                                      dx + r0 * I);
            s->launches += 1;
        }
    }
    return cudaGetLastError();
}

cudaError_t fp32_dw(stacklstm *s, float *dW, float *dbias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H, K = I + H, G = 4 * H;
    const float *dG = (const float *)s->dG;
    if (dW || dbias)
        dw_f32<<<grid_for(s, (size_t)(K + 1) * G, 128), 128, 0, s->stream>>>(
            (size_t)T * B, K, G, (const float *)s->a_rm, dG, dW, dbias);
    if (dW || dbias) s->launches += 1;
    return cudaGetLastError();
}

}  // namespace sl
