// bf16_dev.cuh -- device helpers shared by the bf16 tensor-core kernels (bf16_path.cu,
// bf16_persist.cu): tile constants, the K-major MMA issue of one contraction chunk, the cell
// nonlinearities, vector loads/stores and packing, the step arguments and the forward
// cell epilogue (Algorithm 1: the LSTM cell on the gathered top state, written to history
// row t + 1).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "tc.cuh"

namespace sl {
using tc::smem_u32;
using tc::sw128;

constexpr int kThreads = 128;  // four warps: one per 32-lane quadrant of tensor memory
constexpr int kRows = 128;     // MMA M: batch rows (or weight rows) per CTA tile
constexpr int kChunk = 64;     // contraction elements per chunk: one 128-byte swizzled row
constexpr uint32_t kAStage = kRows * 128;
constexpr int kMaxStages = 16;
constexpr long long kDrainLimit = 4000000000LL;  // wait for own copies / MMAs before exit

// ---- weight packing (one output element each; the forward setup runs all of them in one
// launch, bf16_path.cu)
// Forward operand: for column tile ct, rows n = g * U + j hold gate g of hidden unit
// ct * U + j; each row is the matching column of W over the contraction
// [x padded to 64 ; h padded to 64], in 64-element chunks of 128-byte swizzled rows.
// Element e of [n_ct][KC][4U rows][64].
__device__ __forceinline__ void pack_gate_cols_elem(size_t e, const __nv_bfloat16 *__restrict__ W, int I, int H, int U,
                                                    int kcx, int KC, __nv_bfloat16 *__restrict__ out)
{
    const int NB = 4 * U, G = 4 * H;
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
    const __nv_bfloat16 v = (unit < H && wrow >= 0) ? W[(size_t)wrow * G + g * H + unit] : __float2bfloat16(0.0f);
    const size_t byte = tile * NB * 128 + sw128(row, col >> 3) + (col & 7) * 2;
    out[byte / 2] = v;
}
// Backward operands: for column tile ct, row m is W row (row0 + ct * NB + m) over the 4H
// gate columns (zero padded): W_h rows (row0 = I, rows < I + H) for dh_read, W_x rows
// (row0 = 0, rows < I) for dx. Element e of [n_ct][KC][NB rows][64].
__device__ __forceinline__ void pack_w_rows_elem(size_t e, const __nv_bfloat16 *__restrict__ W, int H, int row0,
                                                 int nrows, int NB, int KC, __nv_bfloat16 *__restrict__ out)
{
    const int G = 4 * H;
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
// Weight chunks of the cluster backward (bf16_cluster.cu): for CTA ct, chunk j, the 16 x 64
// block B[n][16 g + e] = W[I + 16 ct + n][g H + 16 j + e] (zero past H), 128-byte swizzled
// rows. Element e of [n_ct][n_ct chunks][16 rows][64].
constexpr uint32_t kWChunkB = 16 * 128;  // one weight chunk: 16 rows x 64 K
__device__ __forceinline__ void pack_bwd_slice_elem(size_t e, const __nv_bfloat16 *__restrict__ W, int I, int H,
                                                    int n_ct, __nv_bfloat16 *__restrict__ out)
{
    const int kk = (int)(e % 64), nn = (int)((e / 64) % 16);
    const int blk = (int)(e / (64 * 16)), j = blk % n_ct, ct = blk / n_ct;
    const int g = kk / 16, unit = 16 * ct + nn, ku = 16 * j + kk % 16;
    const __nv_bfloat16 v = (unit < H && ku < H) ? W[(size_t)(I + unit) * 4 * H + g * H + ku] : __float2bfloat16(0.0f);
    const uint32_t byte = sw128((uint32_t)nn, (uint32_t)kk >> 3) + (uint32_t)(kk & 7) * 2;
    out[((size_t)blk * kWChunkB + byte) / 2] = v;
}

template <int N>
struct TmemCols {
    static constexpr uint32_t value = N <= 32 ? 32 : N <= 64 ? 64 : N <= 128 ? 128 : 256;
};


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
// The same as one 32-byte access: p must be 32-byte aligned (the fp32 history rows, whose
// length H is a multiple of 8, at a multiple of 8 units).
__device__ __forceinline__ void ld8f_a32(const float *p, float (&v)[8])
{
    asm volatile("ld.global.cg.v8.f32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7])
                 : "l"(p)
                 : "memory");
}
__device__ __forceinline__ void ld8u_a32(const void *p, uint32_t (&w)[8])
{
    asm volatile("ld.global.cg.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7])
                 : "l"(p)
                 : "memory");
}
__device__ __forceinline__ void st8u_a32(void *p, const uint32_t (&w)[8])
{
    asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                 "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}
__device__ __forceinline__ void st8f_a32(float *p, const float (&v)[8])
{
    asm volatile("st.global.v8.f32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "f"(v[0]), "f"(v[1]), "f"(v[2]),
                 "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7])
                 : "memory");
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
    __half *gates;              // [T][B][4H], or (gates_blk) [T][B][H / 16][4][16]
    int gates_blk;              // the blocked gate layout (the cluster forward and backward pair)
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

// ------------------------------------------------------------------ host helpers
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

constexpr uint32_t kSmemCap = 226 * 1024;  // dynamic shared memory; leaves 1 KB for static

template <typename Kern>
cudaError_t allow_smem(Kern k)
{
    return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemCap);
}

// Ring depth: as many stages as the contraction has chunks, within a shared-memory

// ---- persistent step kernels (bf16_persist.cu)
bool bf16_plan_fwd_persist(stacklstm *s, PersistPlan *pl);
bool bf16_plan_bwd_persist(stacklstm *s, PersistPlan *pl);
bool bf16_plan_fwd_cluster(stacklstm *s, PersistPlan *pl);
cudaError_t bf16_launch_fwd_cluster(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_x);
bool bf16_plan_bwd_cluster(stacklstm *s, PersistPlan *pl);
size_t bf16_bwd_cluster_weight_bytes(int H);
cudaError_t bf16_launch_bwd_cluster(stacklstm *s, const StepArgs &a);
cudaError_t bf16_launch_fwd_cluster_group(stacklstm *const *hs, const StepArgs *as, const CUtensorMap *const *tms, int n,
                                          cudaStream_t st);
cudaError_t bf16_launch_bwd_cluster_group(stacklstm *const *hs, const StepArgs *as, int n, cudaStream_t st);
size_t bf16_bwd_cluster_block_bytes(int T, int B, int H);
size_t bf16_fwd_cluster_block_bytes(int T, int B, int H);
cudaError_t bf16_launch_fwd_persist(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_h,
                                    const CUtensorMap &tm_gates, const CUtensorMap &tm_hh,
                                    const CUtensorMap &tm_hc);
cudaError_t bf16_launch_bwd_persist(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_g, float *dx,
                                    bool *dx_done);

// ---- small batches on CUDA cores (bf16_small.cu)
bool bf16_plan_small(stacklstm *s, PersistPlan *pl);
size_t bf16_small_weight_bytes(int I, int H, bool fwd);
cudaError_t bf16_pack_small(stacklstm *s, const __nv_bfloat16 *W);
cudaError_t bf16_launch_fwd_small(stacklstm *s, const StepArgs &a);
cudaError_t bf16_launch_bwd_small(stacklstm *s, const StepArgs &a);

// ---- weight / bias gradients (bf16_dw.cu)
cudaError_t bf16_plan_dw(stacklstm *s);
cudaError_t bf16_launch_dw(stacklstm *s, const CUtensorMap &tm_x, const CUtensorMap &tm_h, const CUtensorMap &tm_g,
                           float *dW, float *dbias);

}  // namespace sl
