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
// The three contractions over all NR = T B rows run on the tensor cores (tcgen05, bf16
// operands, fp32 accumulation; the generic contraction of bf16_path.cu):
//   pre = U Wp^T         U [NR][3H] the gathered tops (zero rows for padding)
//   du  = dP Wp          dP [NR][P] in bf16, scattered into the gradients of the rows read
//   dWp^T = U^T dP       a split contraction over the rows, the parts summed in order
// and the row-wise work on CUDA cores:
//   head_gather    U and each row's (transition, instance, buffer row, label)
//   head_epi       32 rows per CTA: p = ReLU(pre + dp), z, the softmax cross-entropy and
//                  dz, dP = (dz Wz) * (pre > 0); partial sums of dWz, ddp and dq over the
//                  CTA's rows in row order
//   head_scatter   du rows into dy_stack / dy_buffer / dy_action (each output row has one
//                  source row, so plain stores after a zero fill)
//   head_reduce    partial sums in a fixed order: every gradient is bitwise reproducible.
#include <stdio.h>

#include <algorithm>
#include <new>
#include <string>

#include "common.cuh"

struct stacklstm_head {
    int T, Tb, B, H, P, A;
    int device, num_sms;
    cudaStream_t stream;
    int S3;                         // parts of the dWp contraction over the rows
    int NR8;                        // NR rounded up to 8 (row length of U^T)
    __nv_bfloat16 *u = nullptr;     // [NR][3H] gathered tops
    __nv_bfloat16 *ut = nullptr;    // [3H][NR8] the same, transposed
    __nv_bfloat16 *dpb = nullptr;   // [NR][P] dP in bf16
    int4 *meta = nullptr;           // [NR] (k or -1, b, buffer row, label) of each row
    float *pre = nullptr;           // [NR][P] U Wp^T
    float *du = nullptr;            // [NR][3H] dP Wp
    float *part3 = nullptr;         // [S3][3H][P] dWp^T parts
    float *part = nullptr;          // [row blocks][A P + P + A] dWz, ddp, dq partials
    void *wp_k = nullptr, *wpt_k = nullptr, *dpt_k = nullptr;  // packed operands: Wp, Wp^T, dP^T
    float *dh0 = nullptr;           // [2][B][H] gradients of the k = 0 reads (stack, action)
    int32_t *err = nullptr;
    std::string last_error;
};

namespace sl {
namespace {

constexpr int kHeadThreads = 256;
constexpr int kEpiRows = 32;  // rows per head_epi CTA

// One warp per row: the row's transition, instance, buffer row and label (k = -1 for
// padding or a bad length or label, which is recorded), and its U row [s; bu; a].
__global__ void __launch_bounds__(kHeadThreads)
head_gather(int T, int Tb, int B, int H, int A, const __nv_bfloat16 *__restrict__ y_stack,
            const __nv_bfloat16 *__restrict__ h0_stack, const __nv_bfloat16 *__restrict__ y_buffer,
            const __nv_bfloat16 *__restrict__ y_action, const __nv_bfloat16 *__restrict__ h0_action,
            const int32_t *__restrict__ n, const int32_t *__restrict__ L, const int8_t *__restrict__ gold,
            __nv_bfloat16 *__restrict__ u, int4 *__restrict__ meta, int32_t *err)
{
    const int NR = T * B, K = 3 * H, lane = threadIdx.x & 31;
    const int row = blockIdx.x * (kHeadThreads / 32) + (threadIdx.x >> 5);
    if (row >= NR) return;
    const int kk = row / B, b = row % B;
    int k = -1, tb = 0, g = 0;
    const int nb = n[b], Lb = L[b];
    if (kk < Lb) {
        k = kk;
        tb = nb - 1 + kk;
        g = gold[row];
        if (nb < 1 || Lb > T || tb >= Tb || g < 0 || g >= A) {
            if (lane == 0) atomicCAS(err, 0, (int)SL_ERR_ARG);  // the row is skipped
            k = -1;
        }
    }
    if (lane == 0) meta[row] = make_int4(k, b, tb, g);
    for (int pc = lane; pc < K / 8; pc += 32) {
        const int c0 = pc * 8, part = c0 / H, cc = c0 % H;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (k >= 0) {
            const __nv_bfloat16 *src;
            if (part == 0)
                src = k >= 1 ? y_stack + ((size_t)(k - 1) * B + b) * H : h0_stack + (size_t)b * H;
            else if (part == 1)
                src = y_buffer + ((size_t)tb * B + b) * H;
            else
                src = k >= 1 ? y_action + ((size_t)(k - 1) * B + b) * H : h0_action + (size_t)b * H;
            v = *(const uint4 *)(src + cc);
        }
        *(uint4 *)(u + (size_t)row * K + c0) = v;
    }
}

// ut[c][r] = u[r][c] (r < rows), zero for rows .. ld: 32 x 32 tiles through shared memory.
__global__ void head_transpose(const __nv_bfloat16 *__restrict__ u, int rows, int K, int ld,
                               __nv_bfloat16 *__restrict__ ut)
{
    __shared__ __nv_bfloat16 tile[32][33];
    const int r0 = blockIdx.x * 32, c0 = blockIdx.y * 32, tx = threadIdx.x, ty = threadIdx.y;
    for (int i = ty; i < 32; i += blockDim.y) {
        const int r = r0 + i, c = c0 + tx;
        tile[i][tx] = (r < rows && c < K) ? u[(size_t)r * K + c] : __float2bfloat16(0.0f);
    }
    __syncthreads();
    for (int i = ty; i < 32; i += blockDim.y) {
        const int c = c0 + i, r = r0 + tx;
        if (c < K && r < ld) ut[(size_t)c * ld + r] = tile[tx][i];
    }
}

// kEpiRows rows per CTA: p = ReLU(pre + dp), z = Wz p + q, the row's softmax cross-entropy
// and dz, dP = (dz Wz) * (pre > 0) stored in bf16; the CTA's partial sums of dWz [A][P],
// ddp [P] and dq [A] over its rows in row order, to part[blockIdx.x].
__global__ void __launch_bounds__(kHeadThreads)
head_epi(int NR, int P, int A, const float *__restrict__ pre, const float *__restrict__ dp,
         const float *__restrict__ Wz, const float *__restrict__ q, const int4 *__restrict__ meta,
         float *__restrict__ loss_rows, __nv_bfloat16 *__restrict__ dpb, float *__restrict__ part)
{
    extern __shared__ __align__(16) float es[];
    float *p_s = es;                       // [rows][P]
    float *dP_s = p_s + kEpiRows * P;      // [rows][P]
    float *wz_s = dP_s + kEpiRows * P;     // [A][P]
    float *z_s = wz_s + A * P;             // [rows][8]
    float *dz_s = z_s + kEpiRows * 8;      // [rows][8]
    const int tid = threadIdx.x, row0 = blockIdx.x * kEpiRows;
    const int nrow = min(kEpiRows, NR - row0);
    for (int i = tid; i < A * P; i += kHeadThreads) wz_s[i] = Wz[i];
    for (int e = tid; e < kEpiRows * P; e += kHeadThreads) {
        const int r = e / P, j = e % P;
        p_s[e] = r < nrow ? fmaxf(pre[(size_t)(row0 + r) * P + j] + dp[j], 0.0f) : 0.0f;
    }
    __syncthreads();
    // z: warp w takes rows w, w + 8, ...; its lanes split the state columns, then a fixed
    // butterfly sums the lanes
    for (int r = tid >> 5; r < kEpiRows; r += kHeadThreads / 32) {
        const int lane = tid & 31;
        float acc[8];
#pragma unroll
        for (int o = 0; o < 8; ++o) acc[o] = 0.0f;
        for (int j = lane; j < P; j += 32) {
            const float pv = p_s[r * P + j];
#pragma unroll
            for (int o = 0; o < 8; ++o)
                if (o < A) acc[o] = fmaf(wz_s[o * P + j], pv, acc[o]);
        }
#pragma unroll
        for (int o = 0; o < 8; ++o) {
            if (o >= A) break;
            float v = acc[o];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
            if (lane == 0) z_s[r * 8 + o] = v + q[o];
        }
    }
    __syncthreads();
    if (tid < kEpiRows) {
        const int r = tid, row = row0 + r;
        const int4 m = r < nrow ? meta[row] : make_int4(-1, 0, 0, 0);
        float mx = -INFINITY;
        for (int o = 0; o < A; ++o) mx = fmaxf(mx, z_s[r * 8 + o]);
        float sum = 0.0f;
        for (int o = 0; o < A; ++o) sum += __expf(z_s[r * 8 + o] - mx);
        const float lse = mx + __logf(sum);
        const bool valid = m.x >= 0;
        for (int o = 0; o < A; ++o)
            dz_s[r * 8 + o] = valid ? __expf(z_s[r * 8 + o] - lse) - (o == m.w ? 1.0f : 0.0f) : 0.0f;
        if (r < nrow) loss_rows[row] = valid ? lse - z_s[r * 8 + m.w] : 0.0f;
    }
    __syncthreads();
    for (int e = tid; e < kEpiRows * P; e += kHeadThreads) {
        const int r = e / P, j = e % P;
        float acc = 0.0f;
        for (int o = 0; o < A; ++o) acc = fmaf(dz_s[r * 8 + o], wz_s[o * P + j], acc);
        const float d = p_s[e] > 0.0f ? acc : 0.0f;
        dP_s[e] = d;
        if (r < nrow) dpb[(size_t)(row0 + r) * P + j] = __float2bfloat16(d);
    }
    __syncthreads();
    const size_t W = (size_t)A * P + P + A;
    float *pc = part + (size_t)blockIdx.x * W;
    for (int j = tid; j < P; j += kHeadThreads) {
        float aw[8], ad = 0.0f;
#pragma unroll
        for (int o = 0; o < 8; ++o) aw[o] = 0.0f;
        for (int r = 0; r < nrow; ++r) {
            const float pv = p_s[r * P + j];
            ad += dP_s[r * P + j];
#pragma unroll
            for (int o = 0; o < 8; ++o)
                if (o < A) aw[o] = fmaf(dz_s[r * 8 + o], pv, aw[o]);
        }
#pragma unroll
        for (int o = 0; o < 8; ++o)
            if (o < A) pc[(size_t)o * P + j] = aw[o];
        pc[(size_t)A * P + j] = ad;
    }
    if (tid < A) {
        float aq = 0.0f;
        for (int r = 0; r < nrow; ++r) aq += dz_s[r * 8 + tid];
        pc[(size_t)A * P + P + tid] = aq;
    }
}

// du rows into the gradients of the StackLSTM outputs the head read (the k = 0 reads of
// the initial states into dh0); one warp per row, 16-byte pieces.
__global__ void __launch_bounds__(kHeadThreads)
head_scatter(int NR, int B, int H, const float *__restrict__ du, const int4 *__restrict__ meta,
             float *__restrict__ dy_stack, float *__restrict__ dy_buffer, float *__restrict__ dy_action,
             float *__restrict__ dh0)
{
    const int lane = threadIdx.x & 31, row = blockIdx.x * (kHeadThreads / 32) + (threadIdx.x >> 5);
    if (row >= NR) return;
    const int4 m = meta[row];
    const int k = m.x, b = m.y;
    if (k < 0) return;
    const int K = 3 * H;
    for (int pc = lane; pc < K / 4; pc += 32) {
        const int c0 = pc * 4, part = c0 / H, cc = c0 % H;
        float *dst;
        if (part == 0)
            dst = k >= 1 ? dy_stack + ((size_t)(k - 1) * B + b) * H : dh0 + (size_t)b * H;
        else if (part == 1)
            dst = dy_buffer + ((size_t)m.z * B + b) * H;
        else
            dst = k >= 1 ? dy_action + ((size_t)(k - 1) * B + b) * H : dh0 + ((size_t)B + b) * H;
        *(float4 *)(dst + cc) = *(const float4 *)(du + (size_t)row * K + c0);
    }
}

// out[i] = (a0 + a1) + (a2 + a3), a_k the sum over the parts s = k mod 4 in s order; element
// i goes to out0 below n0, else out1 below n0 + n1, else out2. A CTA takes 32 elements (one
// per lane) and its warp k the chain a_k, with 16 loads in flight per pass, so the CTAs of a
// narrow output need not walk all S parts one load at a time.
__global__ void __launch_bounds__(128)
head_reduce(const float *__restrict__ part, int S, size_t n0, size_t n1, size_t n2, float *out0, float *out1,
            float *out2)
{
    __shared__ float chain[4][32];
    const size_t n = n0 + n1 + n2;
    const int lane = threadIdx.x & 31, k = threadIdx.x >> 5;
    const size_t i = blockIdx.x * (size_t)32 + lane;
    float acc = 0.0f;
    if (i < n) {
        int s = k;
        for (; s + 4 * 15 < S; s += 4 * 16) {
            float v[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) v[u] = part[(size_t)(s + 4 * u) * n + i];
#pragma unroll
            for (int u = 0; u < 16; ++u) acc += v[u];
        }
        for (; s < S; s += 4) acc += part[(size_t)s * n + i];
    }
    chain[k][lane] = acc;
    __syncthreads();
    if (k == 0 && i < n) {
        const float a = (chain[0][lane] + chain[1][lane]) + (chain[2][lane] + chain[3][lane]);
        if (i < n0)
            out0[i] = a;
        else if (i < n0 + n1)
            out1[i - n0] = a;
        else
            out2[i - n0 - n1] = a;
    }
}

// dWp [P][K] = the sum over s of the parts of dWp^T [s][K][P], in s order. A CTA (32 x 8
// threads) takes a 32 x 32 tile: its lanes read 32 consecutive j of a part row, each thread
// sums four columns c, and the tile is written transposed through shared memory.
__global__ void __launch_bounds__(256)
head_reduce_t(const float *__restrict__ part, int S, int P, int K, float *__restrict__ dWp)
{
    __shared__ float tile[32][33];  // [c][j]
    const int c0 = blockIdx.x * 32, j0 = blockIdx.y * 32, tx = threadIdx.x, ty = threadIdx.y;
    const int j = j0 + tx;
    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (j < P) {
#pragma unroll 4
        for (int s = 0; s < S; ++s) {
            float v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int c = c0 + ty + 8 * u;
                v[u] = c < K ? part[((size_t)s * K + c) * P + j] : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) acc[u] += v[u];
        }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) tile[ty + 8 * u][tx] = acc[u];
    __syncthreads();
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int jj = j0 + ty + 8 * u, c = c0 + tx;
        if (jj < P && c < K) dWp[(size_t)jj * K + c] = tile[tx][ty + 8 * u];
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

size_t epi_smem(int P, int A) { return ((size_t)2 * kEpiRows * P + (size_t)A * P + 2 * kEpiRows * 8) * 4; }

constexpr long long kHeadWaitLimit = 4000000000LL;  // clock cycles one bounded wait of the contraction may spin

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
    if (H % 8 || P % 8 || P > kHeadThreads || A > 8 || (long long)T * B > (1LL << 30)) return SL_ERR_UNSUPPORTED;
    stacklstm_head *h = new (std::nothrow) stacklstm_head;
    if (!h) return SL_ERR_OOM;
    h->T = T; h->Tb = Tb; h->B = B; h->H = H; h->P = P; h->A = A;
    h->device = device;
    h->stream = (cudaStream_t)stream;
    int prev = -1;
    cudaGetDevice(&prev);
    if (cudaSetDevice(device) != cudaSuccess ||
        cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return SL_ERR_ARG;  // no such device
    }
    const size_t NR = (size_t)T * B, K = 3 * (size_t)H;
    h->NR8 = (int)((NR + 7) / 8 * 8);
    h->S3 = std::max(1, std::min(32, (int)ceil_div(NR, 64) / 8));
    const size_t nblk = ceil_div(NR, kEpiRows), W = (size_t)A * P + P + A;
    auto get = [&](auto **p, size_t bytes) { return cudaMalloc((void **)p, std::max<size_t>(bytes, 16)) == cudaSuccess; };
    bool ok = get(&h->u, NR * K * 2) && get(&h->ut, K * h->NR8 * 2) && get(&h->dpb, NR * P * 2) &&
              get(&h->meta, NR * 16) && get(&h->pre, NR * P * 4) && get(&h->du, NR * K * 4) &&
              get(&h->part3, (size_t)h->S3 * K * P * 4) && get(&h->part, nblk * W * 4) &&
              get(&h->wp_k, bf16_kmajor_bytes(P, (int)K)) && get(&h->wpt_k, bf16_kmajor_bytes((int)K, P)) &&
              get(&h->dpt_k, bf16_kmajor_bytes(P, (int)NR)) && get(&h->dh0, 2 * (size_t)B * H * 4) &&
              get(&h->err, 16);
    if (ok) ok = cudaMemset(h->err, 0, 16) == cudaSuccess;
    if (ok) ok = smem_at_least((const void *)head_epi, epi_smem(P, A)) == cudaSuccess;
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
    const void *vec[] = {y_stack, h0_stack, y_buffer, y_action, h0_action, Wp, dy_stack, dy_buffer, dy_action};
    for (const void *p : vec)
        if (!al16(p)) return head_fail(h, SL_ERR_ARG, "StackLSTM outputs, Wp and dy must be 16-byte aligned");
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    const int T = h->T, B = h->B, H = h->H, P = h->P, A = h->A, K = 3 * H, NR = T * B, sms = h->num_sms;
    const unsigned nblk = ceil_div(NR, kEpiRows), wrows = ceil_div(NR, kHeadThreads / 32);
    const __nv_bfloat16 *wp = (const __nv_bfloat16 *)Wp;
    cudaStream_t st = h->stream;
    cudaError_t e = cudaSuccess;
    // rows of the StackLSTM output gradients the head does not read stay zero
    if (!e) e = cudaMemsetAsync(dy_stack, 0, (size_t)NR * H * 4, st);
    if (!e) e = cudaMemsetAsync(dy_action, 0, (size_t)NR * H * 4, st);
    if (!e) e = cudaMemsetAsync(dy_buffer, 0, (size_t)h->Tb * B * H * 4, st);
    if (!e) e = cudaMemsetAsync(h->dh0, 0, 2 * (size_t)B * H * 4, st);
    // the weights as contraction operands: Wp rows (pre = U Wp^T) and its columns (du = dP Wp)
    if (!e) e = bf16_pack_kmajor(wp, K, false, P, K, h->wp_k, st, sms);
    if (!e) e = bf16_pack_kmajor(wp, K, true, K, P, h->wpt_k, st, sms);
    if (!e) {
        head_gather<<<wrows, kHeadThreads, 0, st>>>(T, h->Tb, B, H, A, (const __nv_bfloat16 *)y_stack,
                                                    (const __nv_bfloat16 *)h0_stack, (const __nv_bfloat16 *)y_buffer,
                                                    (const __nv_bfloat16 *)y_action, (const __nv_bfloat16 *)h0_action,
                                                    n, L, gold, h->u, h->meta, h->err);
        e = cudaGetLastError();
    }
    if (!e) e = bf16_gemm(h->u, K, NR, K, h->wp_k, P, h->pre, 1, st, sms, kHeadWaitLimit, h->err);
    if (!e) {
        head_epi<<<nblk, kHeadThreads, epi_smem(P, A), st>>>(NR, P, A, h->pre, dp, Wz, q, h->meta, loss_rows, h->dpb,
                                                             h->part);
        e = cudaGetLastError();
    }
    if (!e) e = bf16_gemm(h->dpb, P, NR, P, h->wpt_k, K, h->du, 1, st, sms, kHeadWaitLimit, h->err);
    if (!e) {
        head_scatter<<<wrows, kHeadThreads, 0, st>>>(NR, B, H, h->du, h->meta, dy_stack, dy_buffer, dy_action, h->dh0);
        head_transpose<<<dim3(ceil_div(h->NR8, 32), ceil_div(K, 32)), dim3(32, 8), 0, st>>>(h->u, NR, K, h->NR8, h->ut);
        e = cudaGetLastError();
    }
    // dWp^T = U^T dP: a split contraction over the rows, then the parts summed in order
    if (!e) e = bf16_pack_kmajor(h->dpb, P, true, P, NR, h->dpt_k, st, sms);
    if (!e) e = bf16_gemm(h->ut, h->NR8, K, NR, h->dpt_k, P, h->part3, h->S3, st, sms, kHeadWaitLimit, h->err);
    if (!e) {
        head_reduce_t<<<dim3(ceil_div(K, 32), ceil_div(P, 32)), dim3(32, 8), 0, st>>>(h->part3, h->S3, P, K, dWp);
        head_reduce<<<ceil_div((size_t)A * P + P + A, 32), 128, 0, st>>>(h->part, (int)nblk, (size_t)A * P,
                                                                         (size_t)P, (size_t)A, dWz, ddp, dq);
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
    if (v == SL_ERR_TIMEOUT) return head_fail(h, SL_ERR_TIMEOUT, "a device-side wait of a contraction ran out");
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
    void *ps[] = {h->u, h->ut, h->dpb, h->meta, h->pre, h->du, h->part3, h->part, h->wp_k, h->wpt_k, h->dpt_k,
                  h->dh0, h->err};
    for (void *p : ps)
        if (p) cudaFree(p);
    if (prev >= 0) cudaSetDevice(prev);
    delete h;
    return SL_OK;
}

const char *stacklstm_head_last_error(stacklstm_head_t h) { return h ? h->last_error.c_str() : "null handle"; }

}  // extern "C"
