// bf16_cluster.cu -- the forward recurrence (Algorithm 1) for one row tile of at most 64
// instances as a single thread-block cluster. The n_ct column-tile CTAs (16 hidden units
// each, n_ct <= 16) hand each step's h operand to one another through distributed shared
// memory: the epilogue of step t writes its 16 units of h_read(t + 1) (h' where step t
// pushed, else the older top) as one 2 KB slice block to global memory, and one multicast
// bulk copy loads it into every CTA's operand buffer for step t + 1, completing on that
// CTA's mbarrier by byte count. Nothing on the step's critical path goes through global memory
// or a step counter; the history rows, the h operand rows (for the weight gradient) and
// the gates are still written to global memory for the backward.
//
// Warp roles (224 threads): warps 0..3 epilogue (TMEM lane quadrant w, one instance row
// per thread of lanes 0..15; rows >= B idle), warp 4 producer (weight tile once; x_t chunks
// by TMA into a two-step buffer), warps 5 and 6 MMA issue (warp 6: the x part of step t as
// soon as x_t lands; once every slice of h_read(t) has landed, warp 5 the even slices and
// warp 6 the odd ones, each into its own accumulator; accumulators double-buffered by step
// parity).
//
// x_t chunks are 64-row, 128-byte-swizzled 8 KB tiles; an h slice is 16 units x 64 rows in
// the unswizzled K-major core-matrix layout ([row / 8][unit / 8][row mod 8][unit mod 8],
// 2 KB), one K = 16 MMA step. The MMAs are M = 64, the row tile exactly: accumulator rows
// 16 w .. 16 w + 15 sit in lanes 0..15 of TMEM lane quadrant w, so each epilogue warp
// takes 16 rows.
#include <stdio.h>

#include <algorithm>

#include "bf16_dev.cuh"

namespace sl {
namespace {

using tc::smem_u32;

constexpr uint32_t kC64 = 64 * 128;  // one 64-row chunk

struct ClArgs {
    StepArgs s;     // s.kcx: x chunks; s.KC: all chunks
    int n_ct;       // column tiles = CTAs of the cluster
    uint8_t *gscr;  // backward: [T][n_ct] swizzled 8 KB dG blocks
};

// [weight tile KC x NB x 128][h buffers 2 x n_ct x 2 KB][x buffers 2 x kcx x 8 KB][barriers],
// based at the first 1024-byte boundary
constexpr uint32_t kSlice = 2048;
constexpr uint32_t kClBars = 16 * 8 + 16;
__host__ __device__ constexpr uint32_t cl_smem_bytes(int KC, int kcx, int NB, int n_ct)
{
    return 1024 + (uint32_t)KC * NB * 128 + 2u * n_ct * kSlice + 2u * kcx * kC64 + kClBars;
}

struct ClCtl {
    uint32_t w0, h0, x0;  // weight tile, h buffers, x buffers
    uint64_t *wbar, *xfull, *xempty, *hready, *tfull, *tempty, *done;
    uint32_t *tmem_slot;
    volatile int *abort;
};

__device__ __forceinline__ ClCtl cl_carve(uint8_t *raw, int KC, int kcx, int NB, int n_ct)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    ClCtl c;
    const uint32_t wb = (uint32_t)KC * NB * 128, hb = 2u * n_ct * kSlice, xb = 2u * kcx * kC64;
    c.w0 = smem_u32(base);
    c.h0 = c.w0 + wb;
    c.x0 = c.h0 + hb;
    uint64_t *bars = (uint64_t *)(base + wb + hb + xb);
    c.wbar = bars;
    c.xfull = bars + 2;
    c.xempty = bars + 4;
    c.hready = bars + 6;
    c.tfull = bars + 8;
    c.tempty = bars + 10;
    c.done = bars + 12;
    c.tmem_slot = (uint32_t *)(bars + 13);
    c.abort = (volatile int *)(c.tmem_slot + 1);
    return c;
}

__device__ __forceinline__ void cl_abort(const ClCtl &c, int32_t *err)
{
    *c.abort = 1;
    atomicCAS(err, 0, (int)SL_ERR_TIMEOUT);
}

// Bulk copy of `bytes` from global memory into the same shared-memory offset of every CTA
// of cta_mask, completing on the mbarrier at the same offset in each.
__device__ __forceinline__ void bulk_g2s_mc(uint32_t dst, const void *src, uint32_t bytes, uint64_t *bar,
                                            uint16_t cta_mask)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster [%0], [%1], %2, [%3], "
        "%4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "h"(cta_mask)
        : "memory");
}

// Bounded wait (as tc::mbar_wait) with cluster-scope acquire: the phase was completed by
// release arrivals of other CTAs of the cluster, after their distributed-shared-memory stores.
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t *bar, uint32_t parity, long long limit, volatile int *abort)
{
    const long long t0 = clock64();
    while (true) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        if (ok) return true;
        if (clock64() - t0 >= limit) return false;
        if (abort && *abort) return false;
    }
}
// One chunk's four K = 16 MMAs: A (64-row chunk) and the weight chunk (NB rows), K-major,
// 128-byte swizzled.
template <int NB>
__device__ __forceinline__ void cl_mma_chunk(uint32_t d, uint32_t a, uint32_t b, bool first)
{
    constexpr uint32_t idesc = tc::idesc_bf16(NB, 0, 0, 64);
#pragma unroll
    for (int k = 0; k < kChunk / 16; ++k)
        tc::mma_bf16(d, tc::smem_desc(a + k * 32, 16, 1024), tc::smem_desc(b + k * 32, 16, 1024), idesc,
                     !(first && k == 0));
}

// Unswizzled K-major descriptor of an h slice: core matrices (8 rows x 16 bytes) 128 bytes
// apart along K, 256 bytes apart along M.
__device__ __forceinline__ uint64_t slice_desc(uint32_t addr)
{
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)(128 >> 4) << 16) | ((uint64_t)(256 >> 4) << 32) |
           ((uint64_t)1 << 46);
}
// byte offset of 16-byte piece k (units 8k .. 8k + 7) of row r in an h slice
__host__ __device__ constexpr uint32_t slice_off(uint32_t r, uint32_t k) { return (r >> 3) * 256 + k * 128 + (r & 7) * 16; }

// Writes this lane's half of its row of h_read(s) (units 8 h .. 8 h + 7, zero past H or B)
// into its global slice block `blk` (2 KB, the slice layout), then (once every epilogue warp
// has) one multicast bulk copy loads the block into every CTA's h buffer `buf` at this CTA's
// slice position, completing on that CTA's hready[buf]: one L2 read delivered to all CTAs.
__device__ __forceinline__ void deliver_slice(const ClCtl &c, uint8_t *blk, int buf, int row, int h, const uint4 &v,
                                              uint32_t ct, uint32_t n_ct, int tid)
{
    *(uint4 *)(blk + slice_off((uint32_t)row, (uint32_t)h)) = v;
    tc::fence_proxy_async_global();  // this thread's block stores -> the bulk copy
    __syncwarp();
    tc::bar_sync(2, 4 * 32);
    if (tid == 0)
        bulk_g2s_mc(c.h0 + (uint32_t)(buf * n_ct + ct) * kSlice, blk, kSlice, &c.hready[buf],
                    (uint16_t)((1u << n_ct) - 1));
}

constexpr int kClFwdThreads = 224;  // 4 epilogue warps, producer, two MMA issuers

template <int U>
__device__ __forceinline__ void step_cl_body(const CUtensorMap *tmx, const ClArgs &p, int row0)
{
    static_assert(U == 16, "one h slice (two 8-unit core matrices) per CTA");
    constexpr int NB = 4 * U;
    constexpr uint32_t kCols = TmemCols<2 * NB>::value;  // one accumulator per MMA issuer
    constexpr int E = 4;  // epilogue warps
    const StepArgs &a = p.s;
    extern __shared__ uint8_t smem_raw[];
    __shared__ float s_bias[4 * U];
    const int T = a.T, B = a.B, H = a.H, KC = a.KC, kcx = a.kcx;
    const uint32_t ct = tc::cluster_rank(), n_ct = (uint32_t)p.n_ct;
    // this cluster's row tile: rows row0 .. row0 + nrows - 1 of the batch, and its slice blocks
    const int nrows = min(64, B - row0);
    uint8_t *gscr = p.gscr + (size_t)(row0 / 64) * T * n_ct * kSlice;
    const ClCtl c = cl_carve(smem_raw, KC, kcx, NB, (int)n_ct);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const long long limit = a.limit;
    for (int i = tid; i < 4 * U; i += blockDim.x) {
        const int g = i / U, u = (int)ct * U + i % U;
        s_bias[i] = u < H ? a.bias[g * H + u] : 0.0f;
    }
    if (tid == 0) {
        tc::mbar_init(c.wbar, 1);
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&c.xfull[i], 1);
            tc::mbar_init(&c.xempty[i], 1);
            tc::mbar_init(&c.hready[i], 1);
            tc::mbar_init(&c.tfull[i], 2);
            tc::mbar_init(&c.tempty[i], E);
        }
        tc::mbar_init(c.done, 2);
        *c.abort = 0;
        tc::fence_mbar_init();
        // the slices of h_read(0) and h_read(1): every CTA's, by byte count
        for (int t = 0; t < 2 && t < T; ++t) tc::mbar_arrive_expect_tx(&c.hready[t], n_ct * kSlice);
    }
    if (warp == E) tc::tmem_alloc(c.tmem_slot, 2 * kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::cluster_sync();  // every CTA's barriers exist before any copy completes on them
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;

    if (warp == E) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            const uint32_t wbytes = (uint32_t)KC * NB * 128;
            tc::mbar_arrive_expect_tx(c.wbar, wbytes);
            tc::bulk_g2s(c.w0, a.wpack + (size_t)ct * wbytes, wbytes, c.wbar);
            int last = -1;  // last step whose x chunks were issued
            for (int t = 0; t < T && !*c.abort; ++t) {
                const int b = t & 1;
                if (t >= 2 && !tc::mbar_wait(&c.xempty[b], ((t >> 1) - 1) & 1, limit, c.abort)) {
                    cl_abort(c, a.err);
                    break;
                }
                tc::mbar_arrive_expect_tx(&c.xfull[b], (uint32_t)kcx * kC64);
                for (int j = 0; j < kcx; ++j)
                    tc::tma_load_2d(c.x0 + (b * kcx + j) * kC64, tmx, j * kChunk, t * B + row0, &c.xfull[b]);
                last = t;
            }
            // copies still in flight after an abort land before the CTA exits (each buffer's
            // latest phase; phases the MMA warp consumed have completed already)
            for (int t = max(0, last - 1); t <= last; ++t)
                tc::mbar_wait(&c.xfull[t & 1], (t >> 1) & 1, kDrainLimit, nullptr);
        }
        __syncwarp();
    } else if (warp == E + 1 || warp == E + 2) {
        // ------------------------------------------------------------ MMA issue, two issuers
        // The h part (one MMA per slice) is the step's critical path and its MMAs are bound
        // by their issue, so two threads split it, each into its own accumulator (the
        // epilogue adds the two). Issuer 1 also runs the x part, ahead of the h slices,
        // into its accumulator; issuer 0 takes the even slices, issuer 1 the odd ones.
        const int q = warp - (E + 1);
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16(NB, 0, 0, 64);
            bool ok = tc::mbar_wait(c.wbar, 0, limit, c.abort);
            int t_h = -1;  // last step whose h slices all landed
            for (int t = 0; t < T && ok && !*c.abort; ++t) {
                const int b = t & 1;
                if (t >= 2 && !(ok = tc::mbar_wait(&c.tempty[b], ((t >> 1) - 1) & 1, limit, c.abort))) break;
                const uint32_t d = tmem + b * kCols + q * NB;
                if (q == 1) {
                    if (!(ok = tc::mbar_wait(&c.xfull[b], (t >> 1) & 1, limit, c.abort))) break;
                    tc::tc_fence_after();
                    for (int j = 0; j < kcx; ++j)
                        cl_mma_chunk<NB>(d, c.x0 + (b * kcx + j) * kC64, c.w0 + j * NB * 128, j == 0);
                    tc::mma_commit(&c.xempty[b]);
                }
                // the h part once every CTA's slice of h_read(t) has landed
                if (!(ok = mbar_wait_cluster(&c.hready[b], (t >> 1) & 1, limit, c.abort))) break;
                t_h = t;
                // this buffer's next use: its slices cannot land before both issuers have
                // passed this wait (they need this step's MMAs of both)
                if (q == 0 && t + 2 < T) tc::mbar_arrive_expect_tx(&c.hready[b], n_ct * kSlice);
                tc::tc_fence_after();
                const uint32_t hb = c.h0 + (uint32_t)(b * n_ct) * kSlice;
                for (uint32_t j = (uint32_t)q; j < n_ct; j += 2) {
                    const uint32_t k = j * U;  // first h unit of slice j
                    tc::mma_bf16(d, slice_desc(hb + j * kSlice),
                                 tc::smem_desc(c.w0 + (uint32_t)(kcx + k / kChunk) * NB * 128 + (k % kChunk) * 2, 16, 1024),
                                 idesc, q == 1 || j != 0);
                }
                tc::mma_commit(&c.tfull[b]);
            }
            if (!ok) {
                cl_abort(c, a.err);
                // slices other CTAs may still be copying in land before the CTA exits
                if (q == 0)
                    for (int t = t_h + 1; t <= t_h + 2 && t < T; ++t)
                        tc::mbar_wait(&c.hready[t & 1], (t >> 1) & 1, kDrainLimit, nullptr);
            }
            tc::mma_commit(c.done);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        // M = 64 accumulator: rows 16 w .. 16 w + 15 in lanes 0..15 of TMEM lane quadrant w.
        // Two lanes per row: lane l takes row 16 w + l % 16 and units 8 h .. 8 h + 7 of this
        // CTA's 16, h = l / 16; lanes 16..31 take their pre-activations from lane l - 16 by
        // shuffles. Both halves of a row's piece then sit on one line, so every global access
        // of a warp covers its 16 rows in half the L1 wavefronts of one lane per row.
        const int hf = lane >> 4;
        const int row = warp * 16 + (lane & 15);
        const int grow = row0 + row;  // the row of the whole batch
        const bool row_ok = row < nrows;
        const bool warp_rows = warp * 16 < nrows;
        const int u0 = (int)ct * U, uh = u0 + 8 * hf;
        const bool vh = row_ok && uh < H;  // this lane's 8 units (H % 8 == 0)
        const uint32_t taddr0 = tmem + ((uint32_t)(warp * 32) << 16);
        const float *bias_h = s_bias + 8 * hf;  // gate g's bias of this lane's units: bias_h[g U + j]
        // c of the state step t reads, and (when step t does not push) the h of the older
        // state that becomes the next step's h operand
        float crv[8];
        uint4 hold = make_uint4(0u, 0u, 0u, 0u);
        // top[t + 1][row] and top[t + 2][row] at step t (indices loaded two steps ahead)
        int s_nxt = 0, s_2 = 0;
        uint4 h0v = make_uint4(0u, 0u, 0u, 0u);
        if (vh) {
            const int s_cur = a.top[grow];
            s_nxt = T >= 1 ? a.top[(size_t)B + grow] : 0;
            s_2 = T >= 2 ? a.top[(size_t)2 * B + grow] : 0;
            ld8f_a32(a.hist_c + ((size_t)s_cur * B + grow) * H + uh, crv);
            hold = __ldcg((const uint4 *)(a.hr + ((size_t)s_nxt * B + grow) * H + uh));
            h0v = __ldcg((const uint4 *)(a.hr + (size_t)grow * H + uh));  // h_read(0)
        }
        deliver_slice(c, gscr + (size_t)ct * kSlice, 0, row, hf, h0v, ct, n_ct, tid);
        for (int t = 0; t < T; ++t) {
            const int b = t & 1;
            // the next step's operands that rows written before this step hold: issued now,
            // used after this step's cell (c_read of step t + 1 unless step t pushes; the
            // older top that is step t + 2's h operand unless it is this step's new state)
            float cr_n[8];
            uint4 hold_n = make_uint4(0u, 0u, 0u, 0u);
            int s_3 = 0;
            if (vh && t + 1 < T) {
                if (t + 3 <= T) s_3 = a.top[(size_t)(t + 3) * B + grow];
                if (s_nxt != t + 1) ld8f_a32(a.hist_c + ((size_t)s_nxt * B + grow) * H + uh, cr_n);
                if (s_2 <= t) hold_n = __ldcg((const uint4 *)(a.hr + ((size_t)s_2 * B + grow) * H + uh));
            }
            const bool ok = tc::mbar_wait(&c.tfull[b], (t >> 1) & 1, limit, c.abort);
            if (!ok) cl_abort(c, a.err);
            __syncwarp();
            if (tc::bar_any(1, E * 32, !ok || *c.abort)) break;
            tc::tc_fence_after();
            float z[4][8];  // this lane's units of the four gates' pre-activations
            {
                uint32_t zr[4][U];
                if (warp_rows) {
#pragma unroll
                    for (int g = 0; g < 4; ++g) tc::tmem_ld16_async(taddr0 + b * kCols + g * U, zr[g]);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int h2 = 0; h2 < 2; ++h2) {  // the second issuer's accumulator, two gates at a time
                        uint32_t z1[2][U];
#pragma unroll
                        for (int g = 0; g < 2; ++g)
                            tc::tmem_ld16_async(taddr0 + b * kCols + NB + (2 * h2 + g) * U, z1[g]);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int g = 0; g < 2; ++g)
#pragma unroll
                            for (int j = 0; j < U; ++j)
                                zr[2 * h2 + g][j] =
                                    __float_as_uint(__uint_as_float(zr[2 * h2 + g][j]) + __uint_as_float(z1[g][j]));
                    }
                }
                tc::tc_fence_before();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&c.tempty[b]);
#pragma unroll
                for (int g = 0; g < 4; ++g)
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint32_t up = __shfl_sync(0xffffffffu, zr[g][8 + j], lane & 15);
                        z[g][j] = __uint_as_float(hf ? up : zr[g][j]);
                    }
            }
            // the cell (lanes without a row compute and discard)
            float cn[8], hn[8], gv[4][8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float ig = sigm(z[0][j] + bias_h[j]);
                const float fg = sigm(z[1][j] + bias_h[U + j]);
                const float gg = tanh_hw(z[2][j] + bias_h[2 * U + j]);
                const float og = sigm(z[3][j] + bias_h[3 * U + j]);
                cn[j] = fmaf(fg, crv[j], ig * gg);
                hn[j] = og * tanh_hw(cn[j]);
                gv[0][j] = ig; gv[1][j] = fg; gv[2][j] = gg; gv[3][j] = og;
            }
            const bool is_new = s_nxt == t + 1;  // step t pushed: h' is the next step's operand
            const uint4 hb = pack8_bf16(hn), hop = is_new ? hb : hold;
            if (t + 1 < T)
                deliver_slice(c, gscr + ((size_t)(t + 1) * n_ct + ct) * kSlice, (t + 1) & 1, row, hf,
                              vh ? hop : make_uint4(0u, 0u, 0u, 0u), ct, n_ct, tid);
            if (vh) {
                // history row t + 1, the h operand row t + 1 (for the weight gradient), the gates
                const size_t w = ((size_t)(t + 1) * B + grow) * H + uh;
                *(uint4 *)(a.hist_h + w) = hb;
                *(uint4 *)(a.hr + w) = hop;
                st8f_a32(a.hist_c + w, cn);
                // this CTA's 4 x 16 gates of the row: one 128-byte block ([gate][16 units]) or
                // the row-major [4][H] layout
                __half *gt = a.gates_blk ? a.gates + (((size_t)t * B + grow) * n_ct + ct) * 4 * U + 8 * hf
                                         : a.gates + ((size_t)t * B + grow) * 4 * H + uh;
                const size_t gs = a.gates_blk ? (size_t)U : (size_t)H;  // gate stride
#pragma unroll
                for (int g = 0; g < 4; ++g) *(uint4 *)(gt + g * gs) = pack8_f16(gv[g]);
            }
            if (t + 1 < T) {
#pragma unroll
                for (int k = 0; k < 8; ++k) crv[k] = s_nxt == t + 1 ? cn[k] : cr_n[k];
                hold = s_2 == t + 1 ? hb : hold_n;
                s_nxt = s_2;
                s_2 = s_3;
            }
        }
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == E && lane == 0) tc::mbar_wait(c.wbar, 0, kDrainLimit, nullptr);  // after an abort
    if (warp == E + 1 && lane == 0) tc::mbar_wait(c.done, 0, kDrainLimit, nullptr);
    tc::cluster_sync();  // no CTA leaves while another may still copy into its shared memory
    tc::tc_fence_before();
    __syncthreads();
    if (warp == E) tc::tmem_dealloc(tmem, 2 * kCols);
}

constexpr int kClU = 16;        // hidden units per CTA
constexpr int kClMaxTiles = 8;  // row tiles (clusters) of one launch

// ====================================================================== backward
// The reverse-time backward (Sec. 5) for one row tile (B <= 64) as one thread-block
// cluster. Step t multiplies dG_t (all 4H gate columns of the row tile) by this CTA's
// slice of W_h to get dh_read for its 16 units; the epilogue then adds it to the gradient
// of the state step t read and runs the pointwise backward of step t - 1 for its units,
// whose gate gradients dG_{t-1} (4 gates x 16 units x 64 rows) it writes to global memory
// twice: in the [T B][4H] layout (for the input and weight gradients) and as one block of
// 64 rows x 128 bytes (gate-major, 16 units a gate) already in the 128-byte-swizzled
// operand layout, which one multicast bulk copy then loads into every CTA's dG buffer (one
// L2 read of 8 KB, delivered to all CTAs of the cluster, completing on their mbarrier by
// byte count). The K order of the contraction is block order: chunk j is CTA j's block,
// K = 16 g + e for unit 16 j + e of gate g; the weights are packed to match (16 rows x 64,
// 128-byte swizzled, per chunk). The dG buffer is single: before a CTA loads dG_{t-1} in,
// every CTA's step-t MMAs have completed (their commits arrive on the `dfree` barrier of
// every CTA of the cluster). The MMAs are M = 64 (the row tile exactly). The 52 or so
// N = 16 MMAs of a step are bound by their issue, so two threads (warps 4 and 5) issue
// them, each into its own accumulator.
//
// [weight chunks n_ct x 2 KB][dG buffer n_ct x 8 KB][barriers]
// (kWChunkB, one weight chunk of 16 rows x 64 K, and its packing: bf16_dev.cuh)
constexpr uint32_t kGBlock = 64 * 128;   // one CTA's dG block: 64 rows x 64 K
__host__ __device__ constexpr uint32_t clb_smem_bytes(int n_ct)
{
    return 1024 + (uint32_t)n_ct * kWChunkB + (uint32_t)n_ct * kGBlock + kClBars;
}

struct ClbCtl {
    uint32_t w0, g0;  // weight chunks, dG buffer
    uint64_t *wbar, *gready, *dfree, *tfull, *tempty, *done;
    uint32_t *tmem_slot;
    volatile int *abort;
};

__device__ __forceinline__ ClbCtl clb_carve(uint8_t *raw, int n_ct)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    ClbCtl c;
    const uint32_t wb = (uint32_t)n_ct * kWChunkB, gb = (uint32_t)n_ct * kGBlock;
    c.w0 = smem_u32(base);
    c.g0 = c.w0 + wb;
    uint64_t *bars = (uint64_t *)(base + wb + gb);
    c.wbar = bars;
    c.gready = bars + 1;
    c.dfree = bars + 2;
    c.tfull = bars + 3;
    c.tempty = bars + 5;
    c.done = bars + 7;
    c.tmem_slot = (uint32_t *)(bars + 8);
    c.abort = (volatile int *)(c.tmem_slot + 1);
    return c;
}

}  // namespace

namespace {
// One lane's half of a row of a dG block: gate g's units 8 h .. 8 h + 7 (zero past H or B)
// to 16-byte piece 2 g + h of the row in the 128-byte-swizzled global block `blk`.
__device__ __forceinline__ void store_dg_half(uint8_t *blk, int row, int h, const uint4 (&v)[4])
{
#pragma unroll
    for (int g = 0; g < 4; ++g) *(uint4 *)(blk + sw128((uint32_t)row, (uint32_t)(2 * g + h))) = v[g];
}

// After every epilogue warp has stored its rows of the block: thread 0 waits until every
// CTA's MMAs of the step that read the dG buffer completed (dfree phase `fpar`, skipped for
// the first delivery), then loads the block into every CTA's dG buffer at this CTA's chunk.
__device__ __forceinline__ void deliver_dg(const ClbCtl &c, const uint8_t *blk, int fpar, uint32_t ct, uint32_t n_ct,
                                           int tid, long long limit, int32_t *err)
{
    tc::fence_proxy_async_global();  // this thread's block stores -> the bulk copy
    __syncwarp();
    tc::bar_sync(2, 4 * 32);
    if (tid == 0) {
        bool ok = true;
        if (fpar >= 0 && !(ok = mbar_wait_cluster(c.dfree, (uint32_t)fpar, limit, c.abort))) {
            *c.abort = 1;
            atomicCAS(err, 0, (int)SL_ERR_TIMEOUT);
        }
        if (ok) bulk_g2s_mc(c.g0 + ct * kGBlock, blk, kGBlock, c.gready, (uint16_t)((1u << n_ct) - 1));
    }
}

constexpr int kClbIssuers = 4;                          // MMA issue warps
constexpr int kClBwdThreads = (4 + kClbIssuers) * 32;  // and 4 epilogue warps

template <int U>
__device__ __forceinline__ void step_clb_body(const ClArgs &p, int row0)
{
    static_assert(U == 16, "four 16-unit gate slices per CTA");
    constexpr int NI = kClbIssuers;
    static_assert(NI == 2 || NI == 4, "each issuer takes 4 / NI of a chunk's K = 16 steps");
    constexpr uint32_t kCols = TmemCols<NI * U>::value;  // one accumulator per MMA issuer
    constexpr int E = 4;
    const StepArgs &a = p.s;
    extern __shared__ uint8_t smem_raw[];
    const int T = a.T, B = a.B, H = a.H;
    const uint32_t ct = tc::cluster_rank(), n_ct = (uint32_t)p.n_ct;
    // this cluster's row tile: rows row0 .. row0 + nrows - 1 of the batch, and its dG blocks
    const int nrows = min(64, B - row0);
    uint8_t *gscr = p.gscr + (size_t)(row0 / 64) * T * n_ct * kGBlock;
    const ClbCtl c = clb_carve(smem_raw, (int)n_ct);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const long long limit = a.limit;
    if (tid == 0) {
        tc::mbar_init(c.wbar, 1);
        tc::mbar_init(c.gready, 1);
        tc::mbar_init(c.dfree, NI * n_ct);  // every issuer's commits of every CTA
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&c.tfull[i], NI);
            tc::mbar_init(&c.tempty[i], E);
        }
        tc::mbar_init(c.done, NI);
        *c.abort = 0;
        tc::fence_mbar_init();
        tc::mbar_arrive_expect_tx(c.gready, n_ct * kGBlock);  // dG of step T - 1
    }
    if (warp == E) tc::tmem_alloc(c.tmem_slot, 2 * kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::cluster_sync();  // every CTA's barriers exist before any copy or commit lands on them
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;

    if (warp >= E) {
        // ------------------------------------------------------------ MMA issue, NI issuers
        // One thread issues an M = 64, N = 16 MMA about every 45 cycles; two issue about
        // every 30 between them. Issuer q takes the K = 16 steps 4q / NI .. of every chunk
        // into its own accumulator (the epilogue adds them); issuer 0 also posts each
        // step's expected dG bytes and drains, issuer 1 first loads the weights.
        const int q = warp - E;
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16(U, 0, 0, 64);
            if (q == 1) {
                const uint32_t wbytes = n_ct * kWChunkB;
                tc::mbar_arrive_expect_tx(c.wbar, wbytes);
                tc::bulk_g2s(c.w0, a.wpack + (size_t)ct * wbytes, wbytes, c.wbar);
            }
            bool ok = tc::mbar_wait(c.wbar, 0, limit, c.abort);
            int k_g = -1;  // last step index whose dG had landed
            for (int k = 0; k < T && ok && !*c.abort; ++k) {  // step t = T - 1 - k
                const int acc = k & 1;
                if (k >= 2 && !(ok = tc::mbar_wait(&c.tempty[acc], ((k >> 1) - 1) & 1, limit, c.abort))) break;
                if (!(ok = mbar_wait_cluster(c.gready, (uint32_t)(k & 1), limit, c.abort))) break;
                k_g = k;
                // dG of the next step: it cannot land before both issuers have passed this
                // wait (it needs this step's MMAs of both)
                if (q == 0 && k + 1 < T) tc::mbar_arrive_expect_tx(c.gready, n_ct * kGBlock);
                tc::tc_fence_after();
                const uint32_t d = tmem + acc * kCols + q * U;
                for (uint32_t j = 0; j < n_ct; ++j)
#pragma unroll
                    for (int kk = 0; kk < 4 / NI; ++kk) {
                        const int kq = (4 / NI) * q + kk;
                        tc::mma_bf16(d, tc::smem_desc(c.g0 + j * kGBlock + kq * 32, 16, 1024),
                                     tc::smem_desc(c.w0 + j * kWChunkB + kq * 32, 16, 1024), idesc, (j | kk) != 0);
                    }
                tc::mma_commit(&c.tfull[acc]);
                // the dG buffer may be refilled once every CTA's MMAs of this step are done
                tc::mma_commit_mc(c.dfree, (uint16_t)((1u << n_ct) - 1));
            }
            if (!ok) {
                *c.abort = 1;
                atomicCAS(a.err, 0, (int)SL_ERR_TIMEOUT);
                // dG other CTAs may still be copying in lands before the CTA exits
                if (q == 0 && k_g + 1 < T) tc::mbar_wait(c.gready, (uint32_t)((k_g + 1) & 1), kDrainLimit, nullptr);
            }
            tc::mma_commit(c.done);
            // every CTA's commits of the last step have arrived here before the CTA exits
            if (ok && q == 0) mbar_wait_cluster(c.dfree, (uint32_t)((T - 1) & 1), kDrainLimit, nullptr);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        // M = 64 accumulator: rows 16 w .. 16 w + 15 in lanes 0..15 of TMEM lane quadrant w.
        // Two lanes per row: lane l takes row 16 w + l % 16 and units 8 h .. 8 h + 7 of this
        // CTA's 16, h = l / 16; lanes 16..31 take their accumulator values from lane l - 16
        // by shuffles. Both halves of a row's piece then sit on one line, so every global
        // access of a warp covers its 16 rows in half the L1 wavefronts of one lane per row.
        const int hf = lane >> 4;
        const int row = warp * 16 + (lane & 15);
        const int grow = row0 + row;          // the row of the whole batch
        const bool row_ok = row < nrows;
        const bool warp_rows = warp * 16 < nrows;
        const int u0 = (int)ct * U, uh = u0 + 8 * hf;
        const bool vh = row_ok && uh < H;  // this lane's 8 units (H % 8 == 0)
        const uint32_t taddr0 = tmem + ((uint32_t)(warp * 32) << 16);
        const uint4 z4 = make_uint4(0u, 0u, 0u, 0u);
        // dG of step T - 1 (written before the launch) into every CTA's dG buffer
        {
            uint4 g0v[4];
#pragma unroll
            for (int g = 0; g < 4; ++g)
                g0v[g] = vh ? __ldcg((const uint4 *)(a.dG + ((size_t)(T - 1) * B + grow) * 4 * H + g * H + uh)) : z4;
            uint8_t *blk = gscr + ((size_t)(T - 1) * n_ct + ct) * kGBlock;
            store_dg_half(blk, row, hf, g0v);
            deliver_dg(c, blk, -1, ct, n_ct, tid, limit, a.err);
        }
        // the state step t reads (src) and the one step t - 1 read (s1): a step ahead
        int src = 0, s1 = 0;
        if (row_ok) {
            src = a.top[(size_t)(T - 1) * B + grow];
            s1 = T >= 2 ? a.top[(size_t)(T - 2) * B + grow] : 0;
        }
        for (int k = 0; k < T; ++k) {
            const int t = T - 1 - k, acc = k & 1;
            // this step's operands (rows this thread wrote at later steps, or the forward's)
            float dh_src[8], dh_t[8], dc_t[8], cn[8], cr[8], dc_rd[8];
            uint4 gq[4];
            int src_n = 0, s1_n = 0;
            if (row_ok && t >= 1) {
                src_n = a.top[(size_t)(t - 1) * B + grow];
                s1_n = t >= 2 ? a.top[(size_t)(t - 2) * B + grow] : 0;
            }
            if (vh) {
                ld8f_a32(a.dhist_h + ((size_t)src * B + grow) * H + uh, dh_src);
                if (t >= 1) {
                    const size_t wr = ((size_t)t * B + grow) * H + uh, rd = ((size_t)s1 * B + grow) * H + uh;
                    ld8f_a32(a.dhist_h + wr, dh_t);
                    ld8f_a32(a.dhist_c + wr, dc_t);
                    ld8f_a32(a.hist_c + wr, cn);
                    ld8f_a32(a.hist_c + rd, cr);
                    ld8f_a32(a.dhist_c + rd, dc_rd);
                    const __half *gt = a.gates_blk
                                           ? a.gates + (((size_t)(t - 1) * B + grow) * n_ct + ct) * 4 * U + 8 * hf
                                           : a.gates + ((size_t)(t - 1) * B + grow) * 4 * H + uh;
                    const size_t gs = a.gates_blk ? (size_t)U : (size_t)H;  // gate stride
#pragma unroll
                    for (int g = 0; g < 4; ++g) gq[g] = __ldcg((const uint4 *)(gt + g * gs));
                }
            }
            const bool ok = tc::mbar_wait(&c.tfull[acc], (k >> 1) & 1, limit, c.abort);
            if (!ok) {
                *c.abort = 1;
                atomicCAS(a.err, 0, (int)SL_ERR_TIMEOUT);
            }
            __syncwarp();
            if (tc::bar_any(1, E * 32, !ok || *c.abort)) break;
            tc::tc_fence_after();
            float v[8];  // dh_src + the issuers' partial sums, added in issuer order
            {
                float sum[U];
#pragma unroll
                for (int j = 0; j < U; ++j) sum[j] = 0.0f;
                if (warp_rows)
#pragma unroll
                    for (int q2 = 0; q2 < NI; q2 += 2) {
                        uint32_t dr[2][U];
                        tc::tmem_ld16_async(taddr0 + acc * kCols + q2 * U, dr[0]);
                        tc::tmem_ld16_async(taddr0 + acc * kCols + (q2 + 1) * U, dr[1]);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < U; ++j) sum[j] += __uint_as_float(dr[0][j]) + __uint_as_float(dr[1][j]);
                    }
                tc::tc_fence_before();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(&c.tempty[acc]);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float up = __shfl_sync(0xffffffffu, sum[8 + i], lane & 15);
                    v[i] = (hf ? up : sum[i]) + dh_src[i];
                }
            }
            float dcr[8];
            if (t >= 1) {
                // the pointwise backward of step t - 1 (lanes without a row compute and discard)
                float d[4][8], ig[8], fg[8], gg[8], og[8];
                unpack8_f16(gq[0], ig);
                unpack8_f16(gq[1], fg);
                unpack8_f16(gq[2], gg);
                unpack8_f16(gq[3], og);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float dh = src == t ? v[q] : dh_t[q];  // the state read at t is row t
                    const float tcn = tanh_hw(cn[q]);
                    const float dc = dc_t[q] + dh * og[q] * (1.0f - tcn * tcn);
                    d[0][q] = dc * gg[q] * ig[q] * (1.0f - ig[q]);
                    d[1][q] = dc * cr[q] * fg[q] * (1.0f - fg[q]);
                    d[2][q] = dc * ig[q] * (1.0f - gg[q] * gg[q]);
                    d[3][q] = dh * tcn * og[q] * (1.0f - og[q]);
                    dcr[q] = dc_rd[q] + dc * fg[q];
                }
                uint4 dg[4];
#pragma unroll
                for (int g = 0; g < 4; ++g) dg[g] = vh ? pack8_bf16(d[g]) : z4;
                // dG_{t-1}: its block to global memory, then (multicast bulk copy) to every CTA
                uint8_t *blk = gscr + ((size_t)(t - 1) * n_ct + ct) * kGBlock;
                store_dg_half(blk, row, hf, dg);
                deliver_dg(c, blk, k & 1, ct, n_ct, tid, limit, a.err);
                // and in the [T B][4H] layout (for the input and weight gradients), after the delivery
                if (vh) {
                    __nv_bfloat16 *gp = a.dG + ((size_t)(t - 1) * B + grow) * 4 * H + uh;
#pragma unroll
                    for (int g = 0; g < 4; ++g) *(uint4 *)(gp + (size_t)g * H) = dg[g];
                }
            }
            if (vh) {
                st8f_a32(a.dhist_h + ((size_t)src * B + grow) * H + uh, v);
                if (t >= 1) st8f_a32(a.dhist_c + ((size_t)s1 * B + grow) * H + uh, dcr);
            }
            src = src_n;
            s1 = s1_n;
        }
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == E && lane == 0) tc::mbar_wait(c.wbar, 0, kDrainLimit, nullptr);  // after an abort
    if (warp == E + 1 && lane == 0) tc::mbar_wait(c.done, 0, kDrainLimit, nullptr);
    tc::cluster_sync();  // no CTA leaves while another may still copy into its shared memory
    tc::tc_fence_before();
    __syncthreads();
    if (warp == E) tc::tmem_dealloc(tmem, 2 * kCols);
}

// One launch of the forward / backward cluster kernel for one handle.
template <int U>
__global__ void __launch_bounds__(kClFwdThreads, 1) step_cl(const __grid_constant__ CUtensorMap tm_x, ClArgs p)
{
    step_cl_body<U>(&tm_x, p, (int)(blockIdx.x / p.n_ct) * 64);  // cluster m: row tile m
}
template <int U>
__global__ void __launch_bounds__(kClBwdThreads, 1) step_clb(ClArgs p)
{
    step_clb_body<U>(p, (int)(blockIdx.x / p.n_ct) * 64);
}

// Several handles' recurrences in one launch: cluster m (CTAs m n_ct .. m n_ct + n_ct - 1)
// runs member m's steps with its own arguments, workspace and step count. The members are
// independent (each has its own inputs and op stream), so no barrier spans clusters; each
// keeps its own per-step operand exchange.
struct ClGroup {
    CUtensorMap tm[kMaxGroup];  // forward: each member's x map
    ClArgs p[kMaxGroup];
};
template <int U>
__global__ void __launch_bounds__(kClFwdThreads, 1) step_cl_group(const __grid_constant__ ClGroup g)
{
    const int m = (int)blockIdx.x / g.p[0].n_ct;
    step_cl_body<U>(&g.tm[m], g.p[m], 0);
}
template <int U>
__global__ void __launch_bounds__(kClBwdThreads, 1) step_clb_group(const __grid_constant__ ClGroup g)
{
    const int m = (int)blockIdx.x / g.p[0].n_ct;
    step_clb_body<U>(g.p[m], 0);
}

}  // namespace

// Row tiles of 64 instances (instances are independent, so each tile is its own cluster
// of the one launch) up to kClMaxTiles, at most 16 column tiles of 16 units, the footprint
// within the shared-memory cap, and every tile's cluster co-resident on this GPU (a tile
// waiting for SMs would wait for another's whole recurrence); STACKLSTM_FWD_CLUSTER=0
// turns it off (test hook, include/stacklstm.h).
bool bf16_plan_fwd_cluster(stacklstm *s, PersistPlan *pl)
{
    pl->on = 0;
    const char *env = getenv("STACKLSTM_FWD_CLUSTER");
    if (env && atoi(env) == 0) return false;
    const int n_ct = (int)ceil_div(s->H, kClU), tiles = (int)ceil_div(s->B, 64);
    if (tiles > kClMaxTiles || n_ct > 16) return false;
    const int NB = 4 * kClU;
    const uint32_t smem = cl_smem_bytes(s->kcf, s->kcx, NB, n_ct);
    if (smem > kSmemCap) return false;
    const void *fn = (const void *)step_cl<kClU>;
    if (smem_at_least(fn, smem) != cudaSuccess ||
        (n_ct > 8 && cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)) {
        cudaGetLastError();
        return false;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n_ct);
    cfg.blockDim = dim3(kClFwdThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, fn, &cfg) != cudaSuccess || clusters < tiles) {
        cudaGetLastError();
        return false;
    }
    pl->on = 1;
    pl->U = kClU;
    pl->EP = 1;
    pl->n_ct = n_ct;
    pl->cl = n_ct;
    pl->slot = tiles;
    pl->smem = smem;
    pl->threads = kClFwdThreads;
    return true;
}

cudaError_t bf16_launch_fwd_cluster(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_x)
{
    const PersistPlan &pl = s->fc;
    ClArgs p{};
    p.s = a;
    p.s.gates_blk = s->bc.on;  // the cluster backward (and its last-step pointwise) reads the blocked layout
    p.n_ct = pl.n_ct;
    p.gscr = (uint8_t *)s->g_fcl;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.n_ct * pl.slot);  // one cluster per row tile
    cfg.blockDim = dim3(pl.threads);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = s->stream;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = pl.n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, step_cl<kClU>, tm_x, p);
    if (e) return e;
    s->launches += 1;
    return cudaGetLastError();
}

// The backward as one cluster per row tile of 64 instances (as the forward above); at most
// 16 column tiles of 16 units, every tile's cluster co-resident; STACKLSTM_BWD_CLUSTER=0
// turns it off (test hook, include/stacklstm.h). (Copying each CTA's 8 KB of dG into every CTA with bulk copies instead of
// the multicast tensor loads ran 30 % slower than the persistent backward at B = 64,
// H = 200: n_ct^2 copies a step, issued one after another by one thread of each CTA.)
bool bf16_plan_bwd_cluster(stacklstm *s, PersistPlan *pl)
{
    pl->on = 0;
    const char *env = getenv("STACKLSTM_BWD_CLUSTER");
    if (env && atoi(env) == 0) return false;
    const int n_ct = (int)ceil_div(s->H, kClU), tiles = (int)ceil_div(s->B, 64);
    if (tiles > kClMaxTiles || n_ct > 16) return false;
    const uint32_t smem = clb_smem_bytes(n_ct);
    if (smem > kSmemCap) return false;
    const void *fn = (const void *)step_clb<kClU>;
    if (smem_at_least(fn, smem) != cudaSuccess ||
        (n_ct > 8 && cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)) {
        cudaGetLastError();
        return false;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n_ct);
    cfg.blockDim = dim3(kClBwdThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, fn, &cfg) != cudaSuccess || clusters < tiles) {
        cudaGetLastError();
        return false;
    }
    pl->on = 1;
    pl->U = kClU;
    pl->EP = 1;
    pl->n_ct = n_ct;
    pl->cl = n_ct;
    pl->slot = tiles;
    pl->smem = smem;
    pl->threads = kClBwdThreads;
    return true;
}

size_t bf16_fwd_cluster_block_bytes(int T, int B, int H)
{
    return ceil_div(B, 64) * (size_t)T * ceil_div(H, kClU) * kSlice;
}
size_t bf16_bwd_cluster_block_bytes(int T, int B, int H)
{
    return ceil_div(B, 64) * (size_t)T * ceil_div(H, kClU) * kGBlock;
}

size_t bf16_bwd_cluster_weight_bytes(int H)
{
    const size_t n_ct = ceil_div(H, kClU);
    return n_ct * n_ct * kWChunkB;
}

cudaError_t bf16_launch_bwd_cluster(stacklstm *s, const StepArgs &a)
{
    const PersistPlan &pl = s->bc;
    ClArgs p{};
    p.s = a;
    p.s.gates_blk = s->fc.on;  // the cluster forward wrote the blocked layout
    p.n_ct = pl.n_ct;
    p.gscr = (uint8_t *)s->g_bcl;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pl.n_ct * pl.slot);  // one cluster per row tile
    cfg.blockDim = dim3(pl.threads);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = s->stream;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = pl.n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, step_clb<kClU>, p);
    if (e) return e;
    s->launches += 1;
    return cudaGetLastError();
}

// Several handles' forward (or backward) recurrences as one launch of n clusters: the
// dynamic shared memory is the largest member's, each cluster carves its own layout.
template <bool kFwd>
cudaError_t launch_cluster_group(stacklstm *const *hs, const StepArgs *as, const CUtensorMap *const *tms, int n,
                                 cudaStream_t st)
{
    ClGroup g{};
    size_t smem = 0;
    const int n_ct = (kFwd ? hs[0]->fc : hs[0]->bc).n_ct;
    for (int m = 0; m < n; ++m) {
        stacklstm *s = hs[m];
        const PersistPlan &pl = kFwd ? s->fc : s->bc;
        if (!pl.on || pl.n_ct != n_ct || pl.slot != 1) return cudaErrorInvalidValue;
        ClArgs &p = g.p[m];
        p.s = as[m];
        p.s.gates_blk = kFwd ? s->bc.on : s->fc.on;
        p.n_ct = n_ct;
        p.gscr = (uint8_t *)(kFwd ? s->g_fcl : s->g_bcl);
        if (kFwd) g.tm[m] = *tms[m];
        smem = std::max<size_t>(smem, pl.smem);
    }
    const void *fn = kFwd ? (const void *)step_cl_group<kClU> : (const void *)step_clb_group<kClU>;
    cudaError_t e = smem_at_least(fn, smem);
    if (e) return e;
    if (n_ct > 8 && (e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1))) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n * n_ct);
    cfg.blockDim = dim3(kFwd ? kClFwdThreads : kClBwdThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = n_ct;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    void *argv[] = {(void *)&g};
    if ((e = cudaLaunchKernelExC(&cfg, fn, argv))) return e;
    hs[0]->launches += 1;
    return cudaGetLastError();
}

cudaError_t bf16_launch_fwd_cluster_group(stacklstm *const *hs, const StepArgs *as, const CUtensorMap *const *tms, int n,
                                          cudaStream_t st)
{
    return launch_cluster_group<true>(hs, as, tms, n, st);
}

cudaError_t bf16_launch_bwd_cluster_group(stacklstm *const *hs, const StepArgs *as, int n, cudaStream_t st)
{
    return launch_cluster_group<false>(hs, as, nullptr, n, st);
}

}  // namespace sl
