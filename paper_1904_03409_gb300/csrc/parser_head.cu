// parser_head.cu -- the parser head after the three StackLSTMs of a transition-based
// parser (stack, buffer, action history; Sec. 4.1), forward and backward, and its C ABI
// (include/stacklstm.h, stacklstm_head_*).
//
// Before transition k of instance b the head reads the three tops (the output of
// Algorithm 1 of each StackLSTM): s = y_stack[k - 1, b] (h0_stack[b] when k = 0),
// bu = y_buffer[n_b - 1 + k, b] (the buffer was filled by n_b pushes first),
// a = y_action[k - 1, b] (h0_action[b] when k = 0); then p = ReLU(Wp [s; bu; a] + dp)
// (the 200-wide parser state of Sec. 4.1), z = Wz p + q, and the row's loss is
// logsumexp(z) - z[gold]. Rows k >= L_b are padding and contribute nothing.
//
// Kernels (CUDA cores, fp32 accumulation; bf16 inputs):
//   head_rows      R rows (transitions) per CTA: gathers u = [s; bu; a] into shared
//                  memory, pre = u Wp^T + dp, p = ReLU(pre), z, the softmax cross-entropy
//                  and dz, dP = (dz Wz) * (pre > 0), du = dP Wp, and stores du into the
//                  gradients of the StackLSTM outputs (each output row has one source row,
//                  so plain stores after a zero fill); p, dP, dz and u go to the workspace.
//   head_dwp_part  dWp partial sums over one of S row ranges; head_small_part the same for
//                  dWz, ddp and dq; head_reduce sums the partials in range order, so every
//                  gradient is bitwise reproducible.
#include <stdio.h>

#include <string>

#include "common.cuh"

struct stacklstm_head {
    int T, Tb, B, H, P, A, R;
    int device;
    cudaStream_t stream;
    int S;                    // row ranges of the weight-gradient partial sums
    __nv_bfloat16 *wpt = nullptr;  // [3H][P] Wp transposed
    __nv_bfloat16 *u = nullptr;    // [T B][3H] gathered tops
    float *p = nullptr, *dP = nullptr, *dz = nullptr;  // [T B][P], [T B][P], [T B][A]
    float *dh0 = nullptr;     // [2][B][H] gradients of the k = 0 reads (stack, action)
    float *part = nullptr;    // [S][P][3H] dWp partials, then [S2][A P + P + A]
    int32_t *err = nullptr;
    size_t smem = 0;
    std::string last_error;
};

namespace sl {
namespace {

constexpr int kHeadThreads = 256;
constexpr int kSmallChunks = 64;  // row ranges of the dWz / ddp / dq partials
constexpr int kDwpJ = 8;          // Wp rows per dWp CTA

__host__ __device__ constexpr size_t head_smem_bytes(int R, int H, int P, int A)
{
    // u [3H][R] bf16, p [R][P], dP [P][R], Wz [A][P], z and dz [R][A], row info [R]
    return (size_t)3 * H * R * 2 + (size_t)R * P * 4 * 2 + (size_t)A * P * 4 + (size_t)R * A * 4 * 2 + (size_t)R * 16;
}

struct HeadArgs {
    int T, Tb, B, H, P, A;
    const __nv_bfloat16 *y_stack, *h0_stack, *y_buffer, *y_action, *h0_action;
    const int32_t *n, *L;
    const int8_t *gold;
    const __nv_bfloat16 *Wp, *wpt;
    const float *dp, *Wz, *q;
    float *loss_rows, *dy_stack, *dy_buffer, *dy_action, *dh0;
    __nv_bfloat16 *u;
    float *p, *dP, *dz;
    int32_t *err;
};

__global__ void head_pack_wpt(const __nv_bfloat16 *__restrict__ Wp, int P, int K, __nv_bfloat16 *__restrict__ wpt)
{
    const size_t n = (size_t)P * K;
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int j = (int)(e / K), c = (int)(e % K);
        wpt[(size_t)c * P + j] = Wp[e];
    }
}

template <int R>
__global__ void __launch_bounds__(kHeadThreads) head_rows(HeadArgs a)
{
    extern __shared__ __align__(16) uint8_t sm[];
    const int H = a.H, P = a.P, A = a.A, B = a.B, K = 3 * H;
    __nv_bfloat16 *u_s = (__nv_bfloat16 *)sm;                 // [K][R]
    float *p_s = (float *)(sm + (size_t)K * R * 2);           // [R][P]
    float *dP_s = p_s + R * P;                                // [P][R]
    float *wz_s = dP_s + P * R;                               // [A][P]
    float *z_s = wz_s + A * P;                                // [R][A]
    float *dz_s = z_s + R * A;                                // [R][A]
    int *row_k = (int *)(dz_s + R * A);                       // [R] transition, -1 if padding
    int *row_b = row_k + R;
    int *row_tb = row_b + R;                                  // buffer output row read
    int *row_g = row_tb + R;                                  // gold transition
    const int tid = threadIdx.x;
    const int row0 = blockIdx.x * R;
    const int NR = a.T * B;

    for (int i = tid; i < A * P; i += blockDim.x) wz_s[i] = a.Wz[i];
    if (tid < R) {
        const int row = row0 + tid;
        int k = -1, b = 0, tb = 0, g = 0;
        if (row < NR) {
            k = row / B;
            b = row % B;
            const int nb = a.n[b], Lb = a.L[b];
            if (k < Lb) {
                tb = nb - 1 + k;
                g = a.gold[row];
                if (nb < 1 || Lb > a.T || tb >= a.Tb || g < 0 || g >= A) {
                    atomicCAS(a.err, 0, (int)SL_ERR_ARG);  // bad lengths or label: the row is skipped
                    k = -1;
                }
            } else {
                k = -1;
            }
        }
        row_k[tid] = k;
        row_b[tid] = b;
        row_tb[tid] = tb;
        row_g[tid] = g;
    }
    __syncthreads();

    // ---- gather u = [s; bu; a] (16-byte pieces; zeros for padding rows), also to the workspace
    const int pieces = K / 8;
    for (int e = tid; e < R * pieces; e += blockDim.x) {
        const int r = e / pieces, pc = e % pieces, c0 = pc * 8;
        const int k = row_k[r], b = row_b[r];
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (k >= 0) {
            const int part = c0 / H, cc = c0 % H;
            const __nv_bfloat16 *src;
            if (part == 0)
                src = k >= 1 ? a.y_stack + ((size_t)(k - 1) * B + b) * H : a.h0_stack + (size_t)b * H;
            else if (part == 1)
                src = a.y_buffer + ((size_t)row_tb[r] * B + b) * H;
            else
                src = k >= 1 ? a.y_action + ((size_t)(k - 1) * B + b) * H : a.h0_action + (size_t)b * H;
            v = *(const uint4 *)(src + cc);
        }
        if (row0 + r < NR) *(uint4 *)(a.u + (size_t)(row0 + r) * K + c0) = v;
        const __nv_bfloat16 *vh = (const __nv_bfloat16 *)&v;
#pragma unroll
        for (int i = 0; i < 8; ++i) u_s[(size_t)(c0 + i) * R + r] = vh[i];
    }
    __syncthreads();

    // ---- pre = u Wp^T + dp; p = ReLU(pre)   (thread j: column j of all R rows)
    for (int j = tid; j < P; j += blockDim.x) {
        float acc[R];
        const float dpj = a.dp[j];
#pragma unroll
        for (int r = 0; r < R; ++r) acc[r] = dpj;
        for (int c = 0; c < K; ++c) {
            const float w = __bfloat162float(a.wpt[(size_t)c * P + j]);
            const uint4 *ur = (const uint4 *)(u_s + (size_t)c * R);
#pragma unroll
            for (int q8 = 0; q8 < R / 8; ++q8) {
                const uint4 v = ur[q8];
                const __nv_bfloat16 *vh = (const __nv_bfloat16 *)&v;
#pragma unroll
                for (int i = 0; i < 8; ++i) acc[q8 * 8 + i] = fmaf(__bfloat162float(vh[i]), w, acc[q8 * 8 + i]);
            }
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const float pv = fmaxf(acc[r], 0.0f);
            p_s[r * P + j] = pv;
            if (row0 + r < NR) a.p[(size_t)(row0 + r) * P + j] = pv;
        }
    }
    __syncthreads();

    // ---- z = Wz p + q
    for (int t = tid; t < R * A; t += blockDim.x) {
        const int r = t / A, o = t % A;
        float acc = a.q[o];
        for (int j = 0; j < P; ++j) acc = fmaf(wz_s[o * P + j], p_s[r * P + j], acc);
        z_s[t] = acc;
    }
    __syncthreads();

    // ---- softmax cross-entropy of each row and dz
    if (tid < R) {
        const int r = tid, row = row0 + r;
        float m = -INFINITY;
        for (int o = 0; o < A; ++o) m = fmaxf(m, z_s[r * A + o]);
        float s = 0.0f;
        for (int o = 0; o < A; ++o) s += __expf(z_s[r * A + o] - m);
        const float lse = m + __logf(s);
        const bool valid = row_k[r] >= 0;
        for (int o = 0; o < A; ++o) {
            const float d = valid ? __expf(z_s[r * A + o] - lse) - (o == row_g[r] ? 1.0f : 0.0f) : 0.0f;
            dz_s[r * A + o] = d;
            if (row < NR) a.dz[(size_t)row * A + o] = d;
        }
        if (row < NR) a.loss_rows[row] = valid ? lse - z_s[r * A + row_g[r]] : 0.0f;
    }
    __syncthreads();

    // ---- dP = (dz Wz) * (pre > 0)   (thread j)
    for (int j = tid; j < P; j += blockDim.x) {
        for (int r = 0; r < R; ++r) {
            float acc = 0.0f;
            for (int o = 0; o < A; ++o) acc = fmaf(dz_s[r * A + o], wz_s[o * P + j], acc);
            const float d = p_s[r * P + j] > 0.0f ? acc : 0.0f;
            dP_s[j * R + r] = d;
            if (row0 + r < NR) a.dP[(size_t)(row0 + r) * P + j] = d;
        }
    }
    __syncthreads();

    // ---- du = dP Wp, stored into the gradients of the rows the head read
    for (int c = tid; c < K; c += blockDim.x) {
        float acc[R];
#pragma unroll
        for (int r = 0; r < R; ++r) acc[r] = 0.0f;
        for (int j = 0; j < P; ++j) {
            const float w = __bfloat162float(a.Wp[(size_t)j * K + c]);
            const float4 *dr = (const float4 *)(dP_s + (size_t)j * R);
#pragma unroll
            for (int q4 = 0; q4 < R / 4; ++q4) {
                const float4 v = dr[q4];
                acc[4 * q4 + 0] = fmaf(v.x, w, acc[4 * q4 + 0]);
                acc[4 * q4 + 1] = fmaf(v.y, w, acc[4 * q4 + 1]);
                acc[4 * q4 + 2] = fmaf(v.z, w, acc[4 * q4 + 2]);
                acc[4 * q4 + 3] = fmaf(v.w, w, acc[4 * q4 + 3]);
            }
        }
        const int part = c / H, cc = c % H;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = row_k[r], b = row_b[r];
            if (k < 0) continue;
            float *dst;
            if (part == 0)
                dst = k >= 1 ? a.dy_stack + ((size_t)(k - 1) * B + b) * H : a.dh0 + (size_t)b * H;
            else if (part == 1)
                dst = a.dy_buffer + ((size_t)row_tb[r] * B + b) * H;
            else
                dst = k >= 1 ? a.dy_action + ((size_t)(k - 1) * B + b) * H : a.dh0 + ((size_t)B + b) * H;
            dst[cc] = acc[r];
        }
    }
}

// dWp partial sums over row range s: part[s][j][c] = sum over its rows of dP[row][j] u[row][c].
__global__ void __launch_bounds__(kHeadThreads) head_dwp_part(const float *__restrict__ dP,
                                                              const __nv_bfloat16 *__restrict__ u, int NR, int P, int K,
                                                              int S, float *__restrict__ part)
{
    __shared__ float d_s[32][kDwpJ];
    const int tid = threadIdx.x;
    const int j0 = blockIdx.x * kDwpJ, c = blockIdx.y * blockDim.x + tid, s = blockIdx.z;
    const int r_lo = (int)((long long)NR * s / S), r_hi = (int)((long long)NR * (s + 1) / S);
    float acc[kDwpJ];
#pragma unroll
    for (int i = 0; i < kDwpJ; ++i) acc[i] = 0.0f;
    for (int r0 = r_lo; r0 < r_hi; r0 += 32) {
        {
            const int rr = tid / kDwpJ, jj = tid % kDwpJ, row = r0 + rr;
            d_s[rr][jj] = (row < r_hi && j0 + jj < P) ? dP[(size_t)row * P + j0 + jj] : 0.0f;
        }
        __syncthreads();
        const int nr = min(32, r_hi - r0);
        if (c < K)
            for (int rr = 0; rr < nr; ++rr) {
                const float uv = __bfloat162float(u[(size_t)(r0 + rr) * K + c]);
#pragma unroll
                for (int i = 0; i < kDwpJ; ++i) acc[i] = fmaf(d_s[rr][i], uv, acc[i]);
            }
        __syncthreads();
    }
    if (c < K)
#pragma unroll
        for (int i = 0; i < kDwpJ; ++i)
            if (j0 + i < P) part[((size_t)s * P + j0 + i) * K + c] = acc[i];
}

// Partial sums over row range s of dWz [A][P], ddp [P], dq [A]: part[s][A P + P + A].
__global__ void __launch_bounds__(kHeadThreads) head_small_part(const float *__restrict__ p, const float *__restrict__ dP,
                                                                const float *__restrict__ dz, int NR, int P, int A,
                                                                float *__restrict__ part)
{
    const int s = blockIdx.x, S = gridDim.x, tid = threadIdx.x;
    const int r_lo = (int)((long long)NR * s / S), r_hi = (int)((long long)NR * (s + 1) / S);
    const size_t W = (size_t)A * P + P + A;
    for (int j = tid; j < P; j += blockDim.x) {
        float aw[8], ad = 0.0f;
#pragma unroll
        for (int o = 0; o < 8; ++o) aw[o] = 0.0f;
        for (int row = r_lo; row < r_hi; ++row) {
            const float pv = p[(size_t)row * P + j];
            ad += dP[(size_t)row * P + j];
#pragma unroll
            for (int o = 0; o < 8; ++o)
                if (o < A) aw[o] = fmaf(dz[(size_t)row * A + o], pv, aw[o]);
        }
#pragma unroll
        for (int o = 0; o < 8; ++o)
            if (o < A) part[s * W + (size_t)o * P + j] = aw[o];
        part[s * W + (size_t)A * P + j] = ad;
    }
    if (tid < A) {
        float aq = 0.0f;
        for (int row = r_lo; row < r_hi; ++row) aq += dz[(size_t)row * A + tid];
        part[s * W + (size_t)A * P + P + tid] = aq;
    }
}

// out[i] = sum over s of part[s][i], in s order; element i goes to out0 below n0, else
// out1 below n0 + n1, else out2.
__global__ void head_reduce(const float *__restrict__ part, int S, size_t n0, size_t n1, size_t n2, float *out0,
                            float *out1, float *out2)
{
    const size_t n = n0 + n1 + n2;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        float acc = 0.0f;
        for (int s = 0; s < S; ++s) acc += part[(size_t)s * n + i];
        if (i < n0)
            out0[i] = acc;
        else if (i < n0 + n1)
            out1[i - n0] = acc;
        else
            out2[i - n0 - n1] = acc;
    }
}

__global__ void head_add(const float *__restrict__ src, float *a, float *b, size_t n)
{
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        if (a) a[i] += src[i];
        if (b) b[i] += src[n + i];
    }
}

sl_status head_fail(stacklstm_head *h, sl_status st, const char *msg)
{
    if (h) h->last_error = msg;
    return st;
}

sl_status head_cuda(stacklstm_head *h, cudaError_t e, const char *where)
{
    if (h) {
        char buf[256];
        snprintf(buf, sizeof buf, "%s: %s", where, cudaGetErrorString(e));
        h->last_error = buf;
    }
    return SL_ERR_CUDA;
}

bool al16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

unsigned grid_n(size_t n) { return (unsigned)std::max<size_t>(1, std::min<size_t>((n + 255) / 256, 4096)); }

}  // namespace
}  // namespace sl

using namespace sl;

extern "C" {

sl_status stacklstm_head_create(stacklstm_head_t *out, int T, int Tb, int B, int H, int P, int A, int device,
                                void *stream)
{
    if (!out) return SL_ERR_ARG;
    *out = nullptr;
    if (T < 1 || Tb < 1 || B < 1 || H < 1 || P < 1 || A < 2) return SL_ERR_ARG;
    if (H % 8 || P > kHeadThreads || A > 8 || (long long)T * B > (1LL << 30)) return SL_ERR_UNSUPPORTED;
    int R = 32;
    while (R >= 8 && head_smem_bytes(R, H, P, A) > 200 * 1024) R /= 2;
    if (R < 8) return SL_ERR_UNSUPPORTED;
    stacklstm_head *h = new (std::nothrow) stacklstm_head;
    if (!h) return SL_ERR_OOM;
    h->T = T; h->Tb = Tb; h->B = B; h->H = H; h->P = P; h->A = A; h->R = R;
    h->device = device;
    h->stream = (cudaStream_t)stream;
    h->S = std::max(1, std::min(16, (T * B) / 512));
    h->smem = head_smem_bytes(R, H, P, A);
    int prev = -1;
    cudaGetDevice(&prev);
    if (cudaSetDevice(device) != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return SL_ERR_ARG;  // no such device
    }
    const size_t NR = (size_t)T * B, K = 3 * (size_t)H;
    const size_t part = std::max((size_t)h->S * P * K, (size_t)kSmallChunks * ((size_t)A * P + P + A));
    bool ok = cudaMalloc(&h->wpt, K * P * 2) == cudaSuccess && cudaMalloc(&h->u, NR * K * 2) == cudaSuccess &&
              cudaMalloc(&h->p, NR * P * 4) == cudaSuccess && cudaMalloc(&h->dP, NR * P * 4) == cudaSuccess &&
              cudaMalloc(&h->dz, NR * A * 4) == cudaSuccess && cudaMalloc(&h->dh0, 2 * (size_t)B * H * 4) == cudaSuccess &&
              cudaMalloc(&h->part, part * 4) == cudaSuccess && cudaMalloc(&h->err, 16) == cudaSuccess;
    if (ok) ok = cudaMemset(h->err, 0, 16) == cudaSuccess;
    if (ok) {
        const void *fn = R == 32 ? (const void *)head_rows<32> : R == 16 ? (const void *)head_rows<16> : (const void *)head_rows<8>;
        ok = smem_at_least(fn, h->smem) == cudaSuccess;
    }
    if (prev >= 0) cudaSetDevice(prev);
    if (!ok) {
        cudaGetLastError();
        stacklstm_head_destroy(h);
        return SL_ERR_OOM;
    }
    *out = h;
    return SL_OK;
}

sl_status stacklstm_head_run(stacklstm_head_t h, const void *y_stack, const void *h0_stack, const void *y_buffer,
                             const void *y_action, const void *h0_action, const int32_t *n, const int32_t *L,
                             const int8_t *gold, const void *Wp, const float *dp, const float *Wz, const float *q,
                             float *loss_rows, float *dy_stack, float *dy_buffer, float *dy_action, float *dWp,
                             float *ddp, float *dWz, float *dq)
{
    if (!h) return SL_ERR_ARG;
    h->last_error.clear();
    const void *need[] = {y_stack, h0_stack, y_buffer, y_action, h0_action, n, L, gold, Wp, dp, Wz, q,
                          loss_rows, dy_stack, dy_buffer, dy_action, dWp, ddp, dWz, dq};
    for (const void *p : need)
        if (!p) return head_fail(h, SL_ERR_ARG, "null pointer");
    const void *vec[] = {y_stack, h0_stack, y_buffer, y_action, h0_action};
    for (const void *p : vec)
        if (!al16(p)) return head_fail(h, SL_ERR_ARG, "StackLSTM outputs must be 16-byte aligned");
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    const int T = h->T, B = h->B, H = h->H, P = h->P, A = h->A, K = 3 * H;
    const size_t NR = (size_t)T * B;
    cudaStream_t st = h->stream;
    cudaError_t e = cudaSuccess;
    // outputs the row kernel does not write everywhere start at zero
    if (!e) e = cudaMemsetAsync(dy_stack, 0, NR * H * 4, st);
    if (!e) e = cudaMemsetAsync(dy_action, 0, NR * H * 4, st);
    if (!e) e = cudaMemsetAsync(dy_buffer, 0, (size_t)h->Tb * B * H * 4, st);
    if (!e) e = cudaMemsetAsync(h->dh0, 0, 2 * (size_t)B * H * 4, st);
    if (!e) {
        head_pack_wpt<<<grid_n((size_t)P * K), 256, 0, st>>>((const __nv_bfloat16 *)Wp, P, K, h->wpt);
        HeadArgs a;
        a.T = T; a.Tb = h->Tb; a.B = B; a.H = H; a.P = P; a.A = A;
        a.y_stack = (const __nv_bfloat16 *)y_stack; a.h0_stack = (const __nv_bfloat16 *)h0_stack;
        a.y_buffer = (const __nv_bfloat16 *)y_buffer; a.y_action = (const __nv_bfloat16 *)y_action;
        a.h0_action = (const __nv_bfloat16 *)h0_action;
        a.n = n; a.L = L; a.gold = gold;
        a.Wp = (const __nv_bfloat16 *)Wp; a.wpt = h->wpt; a.dp = dp; a.Wz = Wz; a.q = q;
        a.loss_rows = loss_rows; a.dy_stack = dy_stack; a.dy_buffer = dy_buffer; a.dy_action = dy_action;
        a.dh0 = h->dh0; a.u = h->u; a.p = h->p; a.dP = h->dP; a.dz = h->dz; a.err = h->err;
        const unsigned grid = (unsigned)((NR + h->R - 1) / h->R);
        if (h->R == 32)
            head_rows<32><<<grid, kHeadThreads, h->smem, st>>>(a);
        else if (h->R == 16)
            head_rows<16><<<grid, kHeadThreads, h->smem, st>>>(a);
        else
            head_rows<8><<<grid, kHeadThreads, h->smem, st>>>(a);
        head_dwp_part<<<dim3((P + kDwpJ - 1) / kDwpJ, (K + kHeadThreads - 1) / kHeadThreads, h->S), kHeadThreads, 0,
                        st>>>(h->dP, h->u, (int)NR, P, K, h->S, h->part);
        head_reduce<<<grid_n((size_t)P * K), 256, 0, st>>>(h->part, h->S, (size_t)P * K, 0, 0, dWp, nullptr, nullptr);
        e = cudaGetLastError();
    }
    if (!e) {
        // dWz, ddp, dq reuse the partial buffer after dWp's reduction (same stream)
        head_small_part<<<kSmallChunks, kHeadThreads, 0, st>>>(h->p, h->dP, h->dz, (int)NR, P, A, h->part);
        head_reduce<<<grid_n((size_t)A * P + P + A), 256, 0, st>>>(h->part, kSmallChunks, (size_t)A * P, (size_t)P,
                                                                   (size_t)A, dWz, ddp, dq);
        e = cudaGetLastError();
    }
    if (prev >= 0) cudaSetDevice(prev);
    return e ? head_cuda(h, e, "stacklstm_head_run") : SL_OK;
}

sl_status stacklstm_head_add_h0_grads(stacklstm_head_t h, float *dh0_stack, float *dh0_action)
{
    if (!h) return SL_ERR_ARG;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    const size_t n = (size_t)h->B * h->H;
    head_add<<<grid_n(n), 256, 0, h->stream>>>(h->dh0, dh0_stack, dh0_action, n);
    const cudaError_t e = cudaGetLastError();
    if (prev >= 0) cudaSetDevice(prev);
    return e ? head_cuda(h, e, "stacklstm_head_add_h0_grads") : SL_OK;
}

sl_status stacklstm_head_status(stacklstm_head_t h)
{
    if (!h) return SL_ERR_ARG;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    int32_t v = 0;
    cudaError_t e = cudaStreamSynchronize(h->stream);
    if (!e) e = cudaMemcpy(&v, h->err, 4, cudaMemcpyDeviceToHost);
    if (!e && v) e = cudaMemset(h->err, 0, 4);
    if (prev >= 0) cudaSetDevice(prev);
    if (e) return head_cuda(h, e, "stacklstm_head_status");
    if (v) return head_fail(h, (sl_status)v, "a transition with a bad length or label was skipped");
    return SL_OK;
}

sl_status stacklstm_head_destroy(stacklstm_head_t h)
{
    if (!h) return SL_OK;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    if (h->stream) cudaStreamSynchronize(h->stream);
    void *ps[] = {h->wpt, h->u, h->p, h->dP, h->dz, h->dh0, h->part, h->err};
    for (void *p : ps)
        if (p) cudaFree(p);
    if (prev >= 0) cudaSetDevice(prev);
    delete h;
    return SL_OK;
}

const char *stacklstm_head_last_error(stacklstm_head_t h) { return h ? h->last_error.c_str() : "null handle"; }

}  // extern "C"
