// fp32_path.cu -- the fp32 homogenized StackLSTM step on CUDA cores (no tensor cores,
// no TF32). It serves small problems, where B * 4H is too small for a dense tensor-core
// contraction, and is the full-precision counterpart of the bf16 path.
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
#include <algorithm>

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

__global__ void transpose_f32(int R, int C, const float *__restrict__ in, float *__restrict__ out)
{
    const size_t n = (size_t)R * C;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const size_t r = e / C, c = e - r * C;
        out[c * R + r] = in[e];
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

// dh_read = dG_t W_h^T added to row top[t]; grid (ceil(H / blockDim.x), B).
__global__ void bwd_contract_f32(int t, int B, int I, int H, const int32_t *__restrict__ top,
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
    float acc = 0.0f;
    for (int n = 0; n < G; ++n) acc = fmaf(g_s[n], WT[(size_t)n * K + I + k], acc);
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
    for (int n = 0; n < G; ++n) acc = fmaf(g_s[n], WT[(size_t)n * K + k], acc);
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
        for (size_t r = 0; r < R; ++r) {
            const float term = (k < K ? a_rm[r * K + k] : 1.0f) * dG[r * G + n];
            const float y = term - comp;
            const float t = acc + y;
            comp = (t - acc) - y;
            acc = t;
        }
        if (k < K) {
            if (dW) dW[(size_t)k * G + n] = acc;
        } else if (dbias) {
            dbias[n] = acc;
        }
    }
}

unsigned grid_for(const stacklstm *s, size_t n, int threads)
{
    return (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, threads), (size_t)s->num_sms * 32));
}

}  // namespace

cudaError_t fp32_forward_setup(stacklstm *s, const float *h0, const float *c0, const float *W)
{
    const int B = s->B, I = s->I, H = s->H, K = I + H, G = 4 * H;
    cudaError_t e;
    // history row 0 = the initial state (stack slot 0)
    if ((e = cudaMemcpyAsync(s->hist_h, h0, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream))) return e;
    if ((e = cudaMemcpyAsync(s->hist_c, c0, sizeof(float) * B * H, cudaMemcpyDeviceToDevice, s->stream)))
        return e;
    // W^T for the backward contractions (so backward needs nothing the caller owns)
    transpose_f32<<<grid_for(s, (size_t)K * G, 256), 256, 0, s->stream>>>(K, G, W, (float *)s->w_fwd);
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t fp32_forward_steps(stacklstm *s, const float *x, const float *W, const float *bias)
{
    const int T = s->T, B = s->B, I = s->I, H = s->H, K = I + H;
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
    const int threads = std::min(128, ((H + 31) / 32) * 32);
    const unsigned pw_grid = grid_for(s, (size_t)B * H, 256);
    for (int t = T - 1; t >= 0; --t) {
        bwd_pointwise_f32<<<pw_grid, 256, 0, s->stream>>>(t, B, H, s->top, (const float *)s->gates, s->hist_c,
                                                          s->dhist_h, s->dhist_c, dG);
        bwd_contract_f32<<<dim3(ceil_div(H, threads), B), threads, sizeof(float) * G, s->stream>>>(
            t, B, I, H, s->top, WT, dG, s->dhist_h);
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
