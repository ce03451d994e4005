// bf16_dw.cu -- weight and bias gradients of the bf16 path (Sec. 5): dW = sum_t A_t^T dG_t
// with A_t = [x_t ; h_read] and db = sum_{t,b} dG_t, as one split-K contraction over the
// r = t * B + b rows of all steps, reduced in a fixed order (deterministic, no atomics).
//
// Both operands are read MN-major straight from their row-major homes by TMA: x rows (the
// caller's x, [T*B][I]), hr rows (the h operand of each step, [(T+1)*B][H]) and dG rows
// ([T*B][4H]), 64 r-rows per contraction chunk. The M index is padded so that no 64-wide
// block straddles x and h: blocks 0 .. kbx-1 are x columns, kbx .. kbx+kbh-1 are h
// columns, anything after is a constant zero block. A CTA owns MT m (MT / 64 blocks) x 256
// gate columns over a range of chunks: MT = 128, one 256-column accumulator (two CTAs an
// SM), or MT = 256, two accumulators over one shared dG operand (all of tensor memory, one
// CTA an SM, a third fewer operand bytes per MMA). Warps: 0-3 epilogue, 4 TMA producer, 5
// MMA issue. The epilogue warps of the first m tile also sum the dG chunks they find in
// shared memory column by column: the bias gradient, without an all-ones operand row.
#include <stdlib.h>

#include <algorithm>

#include "bf16_dev.cuh"

namespace sl {
namespace {

using tc::smem_u32;
using tc::sw128;

constexpr int kDwThreads = 192;
constexpr int kDwN = 256;            // gate columns per tile
constexpr uint32_t kBlk = 64 * 128;  // one MN-major block: 64 r-rows of 64 bf16 (128 bytes)

struct DwWsArgs {
    int R, I, H;
    int kbx, kbh;  // 64-wide m blocks of x and of h
    int n_nt, split, S;
    float *part;  // [split][rows_part][ld_part]; row rows_part - 1: bias sums
    size_t ld_part, rows_part;
    long long limit;
    int32_t *err;
};

__host__ __device__ constexpr uint32_t dw_stage_bytes(int MT) { return (uint32_t)(MT / 64) * kBlk + kDwN * 128u; }
constexpr uint32_t kDwBarBytes = (2 * kMaxStages + 1) * 8 + 16;
constexpr uint32_t kDwBiasBytes = 128 * 8 * 4;
__host__ __device__ constexpr uint32_t dw_smem_bytes(int S, int MT)
{
    return 1024 + (uint32_t)S * dw_stage_bytes(MT) + kDwBarBytes + kDwBiasBytes;
}

// 8 fp32 values, one whole 32-byte sector (address 32-byte aligned)
__device__ __forceinline__ void st32f(float *p, const float *v)
{
    asm volatile("st.global.v8.f32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "f"(v[0]), "f"(v[1]), "f"(v[2]),
                 "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7])
                 : "memory");
}

template <int MT>
__global__ void __launch_bounds__(kDwThreads, 1)
dw_ws(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_h,
      const __grid_constant__ CUtensorMap tm_g, DwWsArgs a)
{
    constexpr int NT = kDwN;
    constexpr int MB = MT / 64;      // m blocks per tile
    constexpr int NACC = MT / 128;   // accumulators: one per 128 m rows
    constexpr uint32_t kCols = NACC * NT;
    constexpr uint32_t kStage = dw_stage_bytes(MT);
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const int S = a.S;
    const uint32_t ring0 = smem_u32(base);
    uint64_t *full = (uint64_t *)(base + (size_t)S * kStage);
    uint64_t *empty = full + kMaxStages;
    uint64_t *done = empty + kMaxStages;
    uint32_t *tmem_slot = (uint32_t *)(done + 1);
    int *n_issued = (int *)(tmem_slot + 1);
    int *n_consumed = n_issued + 1;
    volatile int *abort = (volatile int *)(n_consumed + 1);
    float *bias_scratch = (float *)((uint8_t *)full + kDwBarBytes);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int mt = blockIdx.x / a.n_nt, nt = blockIdx.x % a.n_nt, sp = blockIdx.y;
    const int RC = (a.R + 63) / 64;
    const int c_lo = (int)((long long)RC * sp / a.split), c_hi = (int)((long long)RC * (sp + 1) / a.split);
    const int KC = c_hi - c_lo;
    const bool do_bias = mt == 0;
    const long long limit = a.limit;
    // kinds of the m blocks: 0 x, 1 h, 2 zero
    int kind[MB], m0[MB];
    for (int j = 0; j < MB; ++j) {
        const int blk = MB * mt + j;
        kind[j] = blk < a.kbx ? 0 : blk < a.kbx + a.kbh ? 1 : 2;
        m0[j] = kind[j] == 0 ? blk * 64 : (blk - a.kbx) * 64;
    }
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(&full[s], 1);
            tc::mbar_init(&empty[s], 1 + (do_bias ? 4 : 0));
        }
        tc::mbar_init(done, 1);
        *n_issued = 0;
        *n_consumed = 0;
        *abort = 0;
        tc::fence_mbar_init();
    }
    // constant zero blocks, in every stage (never overwritten by a copy)
    for (int j = 0; j < MB; ++j)
        if (kind[j] == 2)
            for (int s = 0; s < S; ++s)
                for (uint32_t i = tid; i < kBlk / 16; i += kDwThreads)
                    *(uint4 *)(base + (size_t)s * kStage + j * kBlk + i * 16) = make_uint4(0, 0, 0, 0);
    tc::fence_proxy_async();
    if (warp == 4) tc::tmem_alloc(tmem_slot, kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    auto fail = [&]() {
        *abort = 1;
        atomicCAS(a.err, 0, (int)SL_ERR_TIMEOUT);
    };

    if (warp == 4) {
        if (lane == 0) {
            uint32_t bytes = NT * 128;
            for (int j = 0; j < MB; ++j) bytes += kind[j] != 2 ? kBlk : 0u;
            int it = 0;
            for (; it < KC; ++it) {
                const int s = it % S;
                if (it >= S && !tc::mbar_wait(&empty[s], (uint32_t)(it / S - 1) & 1, limit, abort)) {
                    fail();
                    break;
                }
                const uint32_t st = ring0 + s * kStage;
                const int r0 = (c_lo + it) * 64;
                tc::mbar_arrive_expect_tx(&full[s], bytes);
                for (int j = 0; j < MB; ++j)
                    if (kind[j] != 2) tc::tma_load_2d(st + j * kBlk, kind[j] == 0 ? &tm_x : &tm_h, m0[j], r0, &full[s]);
                for (int nb = 0; nb < NT / 64; ++nb)
                    tc::tma_load_2d(st + MB * kBlk + nb * kBlk, &tm_g, nt * NT + nb * 64, r0, &full[s]);
            }
            *n_issued = it;
        }
        __syncwarp();
    } else if (warp == 5) {
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16(256, 1, 1);
            int it = 0;
            for (; it < KC && !*abort; ++it) {
                const int s = it % S;
                if (!tc::mbar_wait(&full[s], (uint32_t)(it / S) & 1, limit, abort)) {
                    fail();
                    break;
                }
                tc::tc_fence_after();
                const uint32_t as = ring0 + s * kStage, bs = as + MB * kBlk;
#pragma unroll
                for (int k = 0; k < 4; ++k)  // 16 r-rows (two 8-row groups, 2048 bytes) per MMA
#pragma unroll
                    for (int h = 0; h < NACC; ++h)  // m rows 128 h .. + 127: blocks 2 h, 2 h + 1
                        tc::mma_bf16(tmem + h * NT, tc::smem_desc(as + 2 * h * kBlk + k * 2048, kBlk, 1024),
                                     tc::smem_desc(bs + k * 2048, kBlk, 1024), idesc, (it | k) != 0);
                tc::mma_commit(&empty[s]);
            }
            *n_consumed = it;  // chunks whose copies this warp saw land
            tc::mma_commit(done);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------- bias sums
        // column group (8 columns, one 16-byte piece) g of NT / 8, r-rows split tpg ways
        constexpr int NGRP = NT / 8, TPG = 128 / NGRP, RPT = 64 / TPG;
        const int grp = tid % NGRP, sub = tid / NGRP;
        float bsum[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (do_bias) {
            const int nb = grp / 8, q = grp % 8;
            for (int it = 0; it < KC; ++it) {
                const int s = it % S;
                if (!tc::mbar_wait(&full[s], (uint32_t)(it / S) & 1, limit, abort)) {
                    fail();
                    break;
                }
                const uint8_t *blk = base + (size_t)s * kStage + MB * kBlk + nb * kBlk;
#pragma unroll 4
                for (int r = sub * RPT; r < (sub + 1) * RPT; ++r) {
                    const uint4 v = *(const uint4 *)(blk + sw128(r, q));
                    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float2 f = __bfloat1622float2(*(const __nv_bfloat162 *)&w[i]);
                        bsum[2 * i] += f.x;
                        bsum[2 * i + 1] += f.y;
                    }
                }
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&empty[s]);
            }
        }
        // ---------------------------------------------------------- partial sums out
        const bool ok = tc::mbar_wait(done, 0, limit, nullptr);
        if (!ok) fail();
        tc::tc_fence_after();
        if (ok && !*abort) {
#pragma unroll 1
            for (int h = 0; h < NACC; ++h) {
                const size_t m = (size_t)mt * MT + h * 128 + warp * 32 + lane;
                float *dst = a.part + ((size_t)sp * a.rows_part + m) * a.ld_part + (size_t)nt * NT;
                const uint32_t trow = tmem + h * NT + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
                for (int c16 = 0; c16 < NT / 16; ++c16) {
                    float v[16];
                    tc::tmem_ld16(trow + c16 * 16, v);
                    if (KC == 0)
#pragma unroll
                        for (int i = 0; i < 16; ++i) v[i] = 0.0f;
                    st32f(dst + c16 * 16, v);
                    st32f(dst + c16 * 16 + 8, v + 8);
                }
            }
        }
        if (do_bias) {
#pragma unroll
            for (int i = 0; i < 8; ++i) bias_scratch[tid * 8 + i] = bsum[i];
            tc::bar_sync(1, 128);
            if (sub == 0) {
                float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                for (int j = 0; j < TPG; ++j)  // fixed order over the row slices
#pragma unroll
                    for (int i = 0; i < 8; ++i) acc[i] += bias_scratch[(j * NGRP + grp) * 8 + i];
                float *dst = a.part + ((size_t)sp * a.rows_part + a.rows_part - 1) * a.ld_part + (size_t)nt * NT +
                             grp * 8;
                *(float4 *)dst = make_float4(acc[0], acc[1], acc[2], acc[3]);
                *(float4 *)(dst + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
            }
        }
    }
    __syncthreads();
    if (warp == 4 && lane == 0) {
        // copies still in flight after an abort: issued, never seen landed
        for (int it = *n_consumed; it < *n_issued; ++it)
            tc::mbar_wait(&full[it % S], (uint32_t)(it / S) & 1, kDrainLimit, nullptr);
    }
    if (warp == 5 && lane == 0) tc::mbar_wait(done, 0, kDrainLimit, nullptr);
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 4) tc::tmem_dealloc(tmem, kCols);
}

// Fixed-order reduction of the split partials into dW (padded m rows mapped back) and
// dbias (the last partial row).
__global__ void dw_reduce_pad(int I, int H, int kbx, int split, const float *__restrict__ part, size_t rows_part,
                              size_t ld, float *__restrict__ dW, float *__restrict__ dbias)
{
    const int G4 = 4 * H;
    const size_t n = (size_t)(I + H + 1) * (G4 / 4);
    for (size_t e = blockIdx.x * (size_t)blockDim.x + threadIdx.x; e < n; e += (size_t)gridDim.x * blockDim.x) {
        const int m = (int)(e / (G4 / 4)), col = (int)(e % (G4 / 4)) * 4;
        const size_t p = m < I ? (size_t)m : m < I + H ? (size_t)kbx * 64 + (m - I) : rows_part - 1;
        float4 acc = make_float4(0, 0, 0, 0);
        for (int s = 0; s < split; ++s) {
            const float4 v = *(const float4 *)(part + ((size_t)s * rows_part + p) * ld + col);
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
        if (m < I + H) {
            if (dW) *(float4 *)(dW + (size_t)m * G4 + col) = acc;
        } else if (dbias) {
            *(float4 *)(dbias + col) = acc;
        }
    }
}

}  // namespace

// Tile shape, splits and ring depth. 128 x 256 tiles run two CTAs an SM (one's partial-sum
// epilogue overlaps the other's contraction) with a two-stage ring, splits for about two
// waves of such pairs (at least 16 chunks per CTA); their MMAs need about 94 bytes of
// operands a cycle per SM at the full tensor rate, more than TMA delivers (they ran at
// 70-81 % of it). 256 x 256 tiles share one dG operand between two accumulators: one CTA
// an SM, a three-stage ring, and about 62 bytes a cycle. Cost (cycles) = waves x chunks per
// CTA x cycles per chunk (measured) + the split partial sums written and read back at the
// HBM rate; the split count with the least; 512-column tiles and fewer, longer splits
// measured slower. Test hook (include/stacklstm.h): STACKLSTM_DW_M = 128 or 256 fixes the
// tile's m size.
cudaError_t bf16_plan_dw(stacklstm *s)
{
    const int I = s->I, H = s->H, sms = s->num_sms;
    const size_t R = (size_t)s->T * s->B, RC = ceil_div(R, 64);
    const int kbx = (int)ceil_div(I, 64), kbh = (int)ceil_div(H, 64);
    const size_t max_split = std::max<size_t>(1, RC / 16);
    s->dw_ntile = kDwN;
    s->dw_nt = (int)ceil_div(4 * H, kDwN);
    // partial sums of `sp` splits over `rows` padded m rows: written, then read by the reduction
    auto part_cycles = [&](size_t sp, size_t rows) {
        return (double)sp * rows * s->dw_nt * kDwN * 4 * 2 / 6.8e12 * 1.92e9;
    };
    // 128 x 256, two CTAs an SM: splits for about two waves of pairs
    const int mt128 = (kbx + kbh + 1) / 2;
    const size_t tiles128 = (size_t)mt128 * s->dw_nt;
    const size_t split128 = std::min(max_split, std::max<size_t>(1, ceil_div(4 * (size_t)sms, tiles128)));
    const double cost128 = (double)ceil_div(tiles128 * split128, 2 * (size_t)sms) * ceil_div(RC, split128) * 1460.0 +
                           part_cycles(split128, (size_t)mt128 * 128);
    // 256 x 256, one CTA an SM: the split count with the fewest waves x chunks
    const int mt256 = (kbx + kbh + 3) / 4;
    const size_t tiles256 = (size_t)mt256 * s->dw_nt;
    size_t split256 = 1;
    double cost256 = 1e300;
    for (size_t sp = 1; sp <= max_split; ++sp) {
        const double c = (double)ceil_div(tiles256 * sp, (size_t)sms) * ceil_div(RC, sp) * 1140.0 +
                         part_cycles(sp, (size_t)mt256 * 256);
        if (c < cost256 * 0.999) {
            cost256 = c;
            split256 = sp;
        }
    }
    const char *fm = getenv("STACKLSTM_DW_M");
    const bool big = fm ? atoi(fm) == 256 : cost256 < cost128;
    s->dw_mtile = big ? 256 : 128;
    s->dw_mt = big ? mt256 : mt128;
    s->dw_split = (int)(big ? split256 : split128);
    s->sw = big ? 3 : 2;
    s->dw_part_elems = (size_t)s->dw_split * ((size_t)s->dw_mt * s->dw_mtile + 1) * ((size_t)s->dw_nt * kDwN);
    cudaError_t e;
    if ((e = allow_smem(dw_ws<256>)) || (e = allow_smem(dw_ws<128>))) return e;
    return cudaSuccess;
}

cudaError_t bf16_launch_dw(stacklstm *s, const CUtensorMap &tm_x, const CUtensorMap &tm_h, const CUtensorMap &tm_g,
                           float *dW, float *dbias)
{
    DwWsArgs w;
    w.R = s->Tr * s->B;
    w.I = s->I;
    w.H = s->H;
    w.kbx = (int)ceil_div(s->I, 64);
    w.kbh = (int)ceil_div(s->H, 64);
    w.n_nt = s->dw_nt;
    // every split keeps at least 16 chunks of 64 rows (fewer rows than planned: push-only mode)
    w.split = (int)std::min<size_t>(s->dw_split, std::max<size_t>(1, ceil_div((size_t)w.R, 64) / 16));
    w.S = s->sw;
    w.part = s->dw_part;
    w.ld_part = (size_t)s->dw_nt * s->dw_ntile;
    w.rows_part = (size_t)s->dw_mt * s->dw_mtile + 1;
    w.limit = s->wait_limit_bwd;
    w.err = s->err;
    const dim3 grid(s->dw_mt * s->dw_nt, w.split);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kDwThreads);
    cfg.dynamicSmemBytes = dw_smem_bytes(s->sw, s->dw_mtile);
    cfg.stream = s->stream;
    cudaError_t e = s->dw_mtile == 256 ? cudaLaunchKernelEx(&cfg, dw_ws<256>, tm_x, tm_h, tm_g, w)
                                       : cudaLaunchKernelEx(&cfg, dw_ws<128>, tm_x, tm_h, tm_g, w);
    if (e) return e;
    const size_t n = (size_t)(s->I + s->H + 1) * s->H;
    const unsigned blocks = (unsigned)std::max<size_t>(1, std::min<size_t>(ceil_div(n, 256), (size_t)s->num_sms * 16));
    dw_reduce_pad<<<blocks, 256, 0, s->stream>>>(s->I, s->H, w.kbx, w.split, w.part, w.rows_part, w.ld_part, dW,
                                                 dbias);
    s->launches += 2;
    return cudaGetLastError();
}

}  // namespace sl
