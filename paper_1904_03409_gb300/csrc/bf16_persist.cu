// bf16_persist.cu -- persistent, warp-specialised step kernels of the bf16 path: one
// launch (cooperative, or a cluster launch whose clusters all fit at once) runs all T steps
// of the forward (Algorithm 1) or of the reverse-time backward (Sec. 5).
//
// Each CTA keeps one column tile ct (U hidden units: forward, the 4U gate columns of those
// units; backward, U columns of dh_read = dG_t W_h^T) and a fixed set of row tiles
// (rt = slot, slot + n_slot, ...), so every (instance, unit) has one owner for the whole
// launch. Its tiles run in the order (step, rt). The warps have fixed roles:
//   producer (warp 4 EP): loads each tile's A operand by TMA into a ring of S stages of G
//     64-wide contraction chunks (one full / empty mbarrier pair per stage), and the
//     weight tile: once, resident in shared memory, or per stage by bulk copy;
//   MMA (warp 4 EP + 1): waits for a stage, issues its 4G tcgen05.mma (bf16 in, fp32
//     accumulate) in one straight run and commits the stage back. Tiles alternate between
//     two tensor-memory accumulators, so tile k + 1 is multiplied while tile k's epilogue
//     runs. An mbarrier wait between MMAs stalls MMA issue for a few hundred cycles, so a
//     wait covers a whole stage;
//   release (warp 4 EP + 2): raises the row tile's step counter once the epilogue warps
//     have written a tile (its release fence waits for their writes, off their path);
//   epilogue (warps 0 .. 4 EP - 1): warp w reads accumulator lanes 32 (w mod 4) .. + 31
//     (rows) for unit part w / 4. Forward: the LSTM cell, history row t + 1 and the h
//     operand of step t + 1. Backward: adds dh_read to the gradient of the state step t
//     read, then runs the pointwise backward of step t - 1, whose gradient is now complete.
//
// The only inter-CTA dependency is within a row tile: step t reads what every column tile
// of the row tile wrote at the step before (forward: hr[t]; backward: dG_t). Each row tile
// has a counter of completed steps, raised with release semantics after the epilogue's
// stores and polled with acquire semantics (a bounded spin) by the producer before it
// loads the dependent chunks. All CTAs are co-resident (a cooperative launch, or a cluster
// launch whose clusters the planner checked fit at once), so the spins end; every wait is
// bounded and a timeout aborts the whole grid through the error word.
#include <stdio.h>

#include <algorithm>

#include "bf16_dev.cuh"

namespace sl {
namespace {

using tc::smem_u32;

struct WsArgs {
    StepArgs s;              // s.kcx: chunks before the dependent ones; s.S: ring stages
    int n_ct, n_rt, n_slot;  // column tiles (a multiple of cl); row tiles; CTAs per column tile
    int w_res;               // 1: weight tile resident in shared memory
    int32_t *cnt;            // [n_rt] completed steps per row tile (cs ints apart), zero at launch
    int cs;                  // counter stride in ints
    int vec32;               // H % 16 == 0: 16-unit groups of 16-bit rows are 32-byte aligned
    int a_rows;              // rows per A box: 128, or 64 when B <= 64 (one half-filled row tile)
    float *part;             // split contraction: [n_rt][n_ct][KS][128][U] partial dh_read rows
    int32_t *pcnt;           // split contraction: [n_rt][n_ct] partials written, zero at launch
    // backward: CTAs n_chain .. n_chain + n_dx - 1 compute the input gradient alongside the steps
    int n_chain, n_dx;
    int dx_S;                // their ring stages
    int dx_v8;               // dx is 32-byte aligned (whole-sector row stores)
    int nxt;                 // 256-column tiles of dx
    float *dx;               // [T B][I]
    const int32_t *dx_xidx;  // push-only mode: real step of each virtual row's step (-1: none), else null
    const uint8_t *wdx;      // W_x packed as [nxt][KC][256 rows][64], 128-byte swizzled rows
    int cl;                  // 1, or KS: the KS parts of a column tile form a thread-block
                             // cluster and trade their partial sums in shared memory
};

// Dynamic shared memory: [weight tile (w_res)][S stages: G A chunks, then G weight
// chunks unless resident][forward: gate staging tile][split contraction in a cluster:
// partial-sum exchange tile][barriers], based at the first 1024-byte boundary.
constexpr uint32_t kBarBytes = (2 * kMaxStages + 7) * 8 + 32;

// forward: what one tile writes to the history apart from the h operand of the next step,
// staged for the tensor stores that write it out: the activated gates (4 gates x 128 rows
// x U units, fp16), then h' (128 x U, bf16), then c' (128 x U, fp32); each block is laid
// out [unit part][row][units of the part]
// backward with 32-unit tiles: the accumulator rows pass through a [128 rows][32 units]
// fp32 tile on their way from one row per lane to four lanes per row (epilogue_loop)
__host__ __device__ constexpr uint32_t ws_stg_bytes(bool fwd, int U)
{
    return fwd ? 128u * U * (8 + 2 + 4) : U == 32 ? 128u * 32 * 4 : 0u;
}

// split contraction in a cluster: what the other parts send one CTA, fp32 laid out
// [sending part][4-unit group of the U / KS units the CTA finishes][128 rows][4 units]
__host__ __device__ constexpr uint32_t ws_xch_bytes(int U) { return 128u * U * 4; }

__host__ __device__ constexpr uint32_t ws_stage_bytes(int G, int NB, int w_res)
{
    return (uint32_t)G * (kAStage + (w_res ? 0u : (uint32_t)NB * 128));
}
__host__ __device__ constexpr uint32_t ws_smem_bytes(int S, int G, int NB, int KC, int w_res, uint32_t stg)
{
    return 1024 + (w_res ? (uint32_t)KC * NB * 128 : 0u) + (uint32_t)S * ws_stage_bytes(G, NB, w_res) + stg +
           kBarBytes;
}

struct WCtl {
    uint32_t w0, ring0, stage;  // resident weight tile, stage 0, bytes per stage
    uint32_t stg;               // forward: gate staging tile
    uint32_t xch;               // split contraction in a cluster: the partial sums received
    uint64_t *full, *empty, *tfull, *tempty, *wbar, *done;
    uint64_t *rbar;  // one phase per tile: the other parts' partials have landed
    uint32_t *tmem_slot;
    int *n_issued, *n_consumed;  // groups armed by the producer / consumed by the MMA warp
    volatile int *abort;
    volatile int *rel_end;  // tiles the epilogue completed, written before its last barrier with the release warp
};

__device__ __forceinline__ WCtl wcarve(uint8_t *raw, int S, int G, int NB, int KC, int w_res, uint32_t stg,
                                       uint32_t xch)
{
    const uint32_t off = smem_u32(raw);
    uint8_t *base = raw + ((1024u - (off & 1023u)) & 1023u);
    WCtl c;
    const uint32_t wbytes = w_res ? (uint32_t)KC * NB * 128 : 0u;
    c.stage = ws_stage_bytes(G, NB, w_res);
    c.w0 = smem_u32(base);
    c.ring0 = c.w0 + wbytes;
    c.stg = c.ring0 + S * c.stage;
    c.xch = c.stg + stg;
    uint64_t *bars = (uint64_t *)(base + wbytes + (size_t)S * c.stage + stg + xch);
    c.full = bars;
    c.empty = bars + kMaxStages;
    c.tfull = bars + 2 * kMaxStages;
    c.tempty = c.tfull + 2;
    c.wbar = c.tempty + 2;
    c.done = c.wbar + 1;
    c.rbar = c.done + 1;
    c.tmem_slot = (uint32_t *)(c.rbar + 1);
    c.n_issued = (int *)(c.tmem_slot + 1);
    c.n_consumed = c.n_issued + 1;
    c.abort = (volatile int *)(c.n_consumed + 1);
    c.rel_end = c.abort + 1;
    return c;
}

__device__ __forceinline__ void ws_abort(const WCtl &c, int32_t *err)
{
    *c.abort = 1;
    atomicCAS(err, 0, (int)SL_ERR_TIMEOUT);
}

#ifndef STACKLSTM_SPIN_NS
#define STACKLSTM_SPIN_NS 32
#endif
// Bounded spin until *cnt >= target (acquire). False on timeout, on a local abort, or
// once another CTA recorded an error.
__device__ __forceinline__ bool spin_until(const int32_t *cnt, int target, long long limit, volatile int *abort,
                                           const int32_t *err, unsigned sleep_ns = STACKLSTM_SPIN_NS)
{
    if (tc::ld_acquire_gpu(cnt) >= target) return true;
    const long long t0 = clock64();
    while (true) {
        if (clock64() - t0 >= limit) return false;
        if (*abort || *(const volatile int32_t *)err) return false;
        __nanosleep(sleep_ns);
        if (tc::ld_acquire_gpu(cnt) >= target) return true;
    }
}

// One stage's MMAs: n (<= G) chunks of four K = 16 steps, K-major operands in 128-byte
// swizzled rows (A chunks kAStage apart, weight chunks NB * 128 bytes apart).
template <int NB, int G>
__device__ __forceinline__ void issue_group(uint32_t d, uint32_t a, uint32_t b, int n, bool first)
{
    constexpr uint32_t idesc = tc::idesc_bf16(NB);
#pragma unroll
    for (int j = 0; j < G; ++j)
        if (j < n) {
#pragma unroll
            for (int k = 0; k < kChunk / 16; ++k)
                tc::mma_bf16(d, tc::smem_desc(a + j * kAStage + k * 32, 16, 1024),
                             tc::smem_desc(b + j * (NB * 128) + k * 32, 16, 1024), idesc,
                             !(first && j == 0 && k == 0));
        }
}

// Loads UE consecutive accumulator columns of this thread's lane (no completion wait).
template <int UE>
__device__ __forceinline__ void tmem_cols(uint32_t taddr, uint32_t (&r)[UE])
{
    if constexpr (UE % 16 == 0) {
#pragma unroll
        for (int i = 0; i < UE / 16; ++i) tc::tmem_ld16_async(taddr + i * 16, *(uint32_t(*)[16])(r + i * 16));
    } else {
#pragma unroll
        for (int i = 0; i < UE / 8; ++i) tc::tmem_ld8_async(taddr + i * 8, *(uint32_t(*)[8])(r + i * 8));
    }
}

// chunk range of the stage that starts at chunk c0: never mixes the independent chunks
// (< split) with the dependent ones
__device__ __forceinline__ int group_end(int c0, int G, int split, int KC)
{
    return min(c0 + G, c0 < split ? split : KC);
}

// ------------------------------------------------------------- vector access
#ifndef LD_V8_OP
#define LD_V8_OP "ld.global.cg.v8.b32"
#endif
// NG (8 or 16) consecutive values of one row per thread: 16- or 32-byte accesses, so a
// lane fills whole 32-byte L2 sectors where the row layout allows (fp32: always; 16-bit
// rows: when H is a multiple of 16). Addresses are NG * element size aligned.
__device__ __forceinline__ void st_v8(void *p, const uint32_t *w)
{
    asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                 "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
}
__device__ __forceinline__ void ld_v8(const void *p, uint32_t *w)
{
    asm volatile(LD_V8_OP " {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7])
                 : "l"(p)
                 : "memory");
}
__device__ __forceinline__ void st_v4(void *p, const uint32_t *w)
{
    *(uint4 *)p = make_uint4(w[0], w[1], w[2], w[3]);
}
__device__ __forceinline__ void ld_v4(const void *p, uint32_t *w)
{
    const uint4 v = __ldcg((const uint4 *)p);
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
}
__device__ __forceinline__ void ld_shared_v4(uint32_t addr, uint32_t *w)
{
    asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]) : "r"(addr));
}
// NG 16-bit values (raw words, NG / 2 of them)
template <int NG>
__device__ __forceinline__ void st_h(void *p, const uint32_t *w)
{
    if constexpr (NG == 16) st_v8(p, w); else st_v4(p, w);
}
template <int NG>
__device__ __forceinline__ void ld_h(const void *p, uint32_t *w)
{
    if constexpr (NG == 16) ld_v8(p, w); else ld_v4(p, w);
}
// NG fp32 values (32-byte pieces)
template <int NG>
__device__ __forceinline__ void st_f(float *p, const float *v)
{
#pragma unroll
    for (int i = 0; i < NG / 8; ++i) st_v8(p + 8 * i, (const uint32_t *)(v + 8 * i));
}
template <int NG>
__device__ __forceinline__ void ld_f(const float *p, float *v)
{
#pragma unroll
    for (int i = 0; i < NG / 8; ++i) ld_v8(p + 8 * i, (uint32_t *)(v + 8 * i));
}
template <int NG>
__device__ __forceinline__ void pack_bf16(const float *v, uint32_t *w)
{
#pragma unroll
    for (int i = 0; i < NG / 2; ++i) {
        __nv_bfloat162 t = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *(uint32_t *)&t;
    }
}
template <int NG>
__device__ __forceinline__ void pack_f16(const float *v, uint32_t *w)
{
#pragma unroll
    for (int i = 0; i < NG / 2; ++i) {
        __half2 t = __floats2half2_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *(uint32_t *)&t;
    }
}
template <int NG>
__device__ __forceinline__ void unpack_f16(const uint32_t *w, float *v)
{
#pragma unroll
    for (int i = 0; i < NG / 2; ++i) {
        const float2 f = __half22float2(*(const __half2 *)&w[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// L2 prefetch of one row piece: the line holding its start. (Measured slower: a prefetch
// per 32-byte sector, and bulk-engine prefetches of the whole piece, which queue behind
// the ring's tensor copies.)
__device__ __forceinline__ void pf_l2(const void *p, uint32_t) { tc::prefetch_l2(p); }

// Backward: store the gradient-history updates after the step's release, so that the
// release (and the proxy fence before it) does not wait for them. Their values stay in
// registers meanwhile: done with one epilogue warp group (6 warps, up to 255 registers a
// thread), not with two (10 warps share the register file: 168 a thread, and the held
// values spill; measured slower).
#ifndef STACKLSTM_DEFER_DHIST
#define STACKLSTM_DEFER_DHIST 1
#endif
template <int EP>
__host__ __device__ constexpr bool defer_dhist() { return STACKLSTM_DEFER_DHIST != 0 && EP == 1; }

// Byte offset of 16-byte piece q of row r in a staging tile of RB-byte rows, in the layout
// the tensor map's swizzle mode (32, 64 or 128 bytes for rows of that size; none for
// 16-byte rows) gives the tile: the offset's 16-byte-piece bits XOR its 128-byte-line bits,
// over log2(RB / 16) bits. Lanes that write one row each then hit distinct banks.
template <int RB>
__device__ __forceinline__ uint32_t stg_swz(uint32_t r, uint32_t q)
{
    static_assert(RB == 16 || RB == 32 || RB == 64 || RB == 128, "staging rows of 16 to 128 bytes");
    const uint32_t o = r * RB + q * 16;
    return o ^ (((o >> 7) & (RB / 16 - 1)) << 4);
}

// ------------------------------------------------------------------ epilogue
// Named barrier of the epilogue warps with the release warp, once a tile. The release
// (`red.release.gpu`) waits for every earlier memory operation to be performed, about
// 1.4-1.8 K cycles. The backward whose epilogue is its bottleneck (32-unit tiles, four lanes
// a row, several row tiles a CTA) hands it to a warp of its own, off the epilogue's path
// (-4.7 %). Elsewhere thread 0 of the epilogue releases: there the counter is on the step
// chain, and the fence of a separate warp also waited for the stores and loads the
// epilogue issued after the barrier (large backward +5.6 %, stress forward +6 %).
constexpr int kRelBar = 4;
template <int U, int EP, bool kFwd, int KS>
__host__ __device__ constexpr bool rel_warp_variant()
{
    return !kFwd && KS == 1 && EP == 1 && U == 32 && defer_dhist<EP>();
}
// the same for every thread of the launch: that variant, with more row tiles than slots
template <int U, int EP, bool kFwd, int KS>
__device__ __forceinline__ bool rel_warp(const WsArgs &p)
{
    return rel_warp_variant<U, EP, kFwd, KS>() && p.n_rt > p.n_slot;
}

struct EpiCtx {
    WCtl c;
    uint32_t tmem;
    int q, part, lane, tid;  // TMEM lane quadrant, unit part, lane, thread
    int ct, kp, slot, n_mine, n_tiles;  // column tile, contraction part, slot
    long long limit;
};

// All tiles of one epilogue thread: row 32 q + lane of each tile, in access groups of NG
// units. Without a split contraction (KS = 1) the thread finishes units
// ct * U + part * UE .. + UE straight from its accumulator lane. With KS > 1 (backward
// only) the KS CTAs of a column tile each hold a partial dh_read over a quarter (half ...)
// of the 4H contraction and finish U / KS units, ct * U + kp * U / KS .. + U / KS, summing
// the parts in part order (deterministic). The parts trade their partials as one
// thread-block cluster, each storing the other parts' units of its row into their shared
// memory (p.cl = KS), or through an L2 scratch: every CTA writes its whole partial row,
// counts it, waits for the other parts and reads back its units of each.
template <int U, int EP, int NG, bool kFwd, int KS>
__device__ __forceinline__ void epilogue_loop(const StepArgs &a, const WsArgs &p, const EpiCtx &e,
                                              const float *s_bias, const CUtensorMap *tm_gates,
                                              const CUtensorMap *tm_hh, const CUtensorMap *tm_hc)
{
    static_assert(KS == 1 || (!kFwd && EP == 1), "split contraction: backward, one epilogue warp group");
    constexpr int E = 4 * EP, UE = U / KS / EP;  // units this thread finishes
    constexpr int NB = kFwd ? 4 * U : U;
    constexpr uint32_t kCols = TmemCols<NB>::value;
    const int T = a.T, B = a.B, H = a.H;
    const uint32_t lane_off = (uint32_t)(e.q * 32) << 16;
    const int u0 = e.ct * U + e.kp * (U / KS) + e.part * UE;  // first unit of this thread
    // The row indices of a tile for this thread: the state it reads (src) and, forward, the
    // top after the step (s_next) / backward, the state step t - 1 read (s1). They are
    // loaded a tile ahead, so that no load waits on another at the start of a tile.
    auto tile_rows = [&](int kk, int &i0, int &i1) {
        const int ksk = kk / e.n_mine, rtk = e.slot + (kk % e.n_mine) * p.n_slot;
        const int tk = kFwd ? ksk : T - 1 - ksk;
        const int bk = rtk * kRows + e.q * 32 + e.lane;
        i0 = 0;
        i1 = 0;
        if (bk < B) {
            i0 = a.top[(size_t)tk * B + bk];
            if (kFwd)
                i1 = a.top[(size_t)(tk + 1) * B + bk];
            else if (tk >= 1)
                i1 = a.top[(size_t)(tk - 1) * B + bk];
        }
    };
    int cur0 = 0, cur1 = 0;
    if (e.n_tiles > 0) tile_rows(0, cur0, cur1);
    constexpr bool kLatePfBwd = UE > 16;  // backward: operands taken group by group (below)
    // backward, 32 units a thread, unsplit contraction: four lanes per row (below)
    constexpr bool kRows4 = !kFwd && KS == 1 && EP == 1 && UE == 32 && defer_dhist<EP>();
    int k = 0;
    for (; k < e.n_tiles; ++k) {
        const int ks = k / e.n_mine, rt = e.slot + (k % e.n_mine) * p.n_slot;
        const int t = kFwd ? ks : T - 1 - ks;
        const int b = rt * kRows + e.q * 32 + e.lane;
        const bool row_ok = b < B;
        const int acc = k & 1;
        const uint32_t taddr = e.tmem + acc * kCols + lane_off;
        int nx0 = 0, nx1 = 0;
        if (k + 1 < e.n_tiles) tile_rows(k + 1, nx0, nx1);
        const bool pf_early = e.n_mine == 1;  // forward; the backward decides by its tile shape
        // the next tile's epilogue operands into L2 (their loads then wait on L2, not HBM).
        // Forward with one row tile per CTA, and backward with one access group a thread:
        // prefetched as soon as this tile's own loads are issued (waiting for the indices);
        // else once this tile's work is done (the indices have arrived; the forward's next
        // tile is another row tile's). Measured per shape. A row the current tile is about
        // to write is harmless to prefetch.
        auto prefetch_next = [&]() {
            if (k + 1 >= e.n_tiles) return;
            const int ks1 = (k + 1) / e.n_mine, rt1 = e.slot + ((k + 1) % e.n_mine) * p.n_slot;
            const int t1 = kFwd ? ks1 : T - 1 - ks1;
            const int b1 = rt1 * kRows + e.q * 32 + e.lane;
            if (b1 >= B || u0 >= H) return;
            // this thread's whole row pieces (H and u0 are multiples of 8: 16-byte aligned,
            // whole 16-byte multiples)
            const uint32_t n4 = 4u * (uint32_t)min(UE, H - u0), n2 = n4 / 2;
            if constexpr (kFwd) {
                pf_l2(a.hist_c + ((size_t)nx0 * B + b1) * H + u0, n4);
                pf_l2(a.hr + ((size_t)nx1 * B + b1) * H + u0, n2);
            } else {
                pf_l2(a.dhist_h + ((size_t)nx0 * B + b1) * H + u0, n4);
                if (t1 >= 1) {
                    const size_t wr = ((size_t)t1 * B + b1) * H + u0, rd = ((size_t)nx1 * B + b1) * H + u0;
                    pf_l2(a.dhist_h + wr, n4);
                    pf_l2(a.dhist_c + wr, n4);
                    pf_l2(a.hist_c + wr, n4);
                    pf_l2(a.hist_c + rd, n4);
                    pf_l2(a.dhist_c + rd, n4);
                    const __half *gt = a.gates + ((size_t)(t1 - 1) * B + b1) * 4 * H + u0;
#pragma unroll
                    for (int g = 0; g < 4; ++g) pf_l2(gt + (size_t)g * H, n2);
                }
            }
        };
        // backward: the gradient-history rows this thread updates, stored after the step's
        // release (only this thread reads them again, at later steps)
        constexpr bool kDeferDhist = !kFwd && defer_dhist<EP>();
        float dfh[kDeferDhist ? UE : 1], dfc[kDeferDhist ? UE : 1];
        int d_src = 0, d_s1 = 0;
        // four lanes per row (below): the rows' history indices, by round
        int r_src[kRows4 ? 4 : 1], r_s1[kRows4 ? 4 : 1];
        bool r_ok[kRows4 ? 4 : 1];
        if constexpr (kFwd) {
            // operands this thread wrote itself at earlier steps (same rows and units):
            // c_read, and the older top the next step reads when step t does not push
            const int src = cur0, s_next = cur1;
            const bool is_new = s_next == t + 1;
            float cr[UE];
            uint32_t hc[UE / 2];
            if (k >= e.n_mine) {
                // c' leaves by tensor store: the stores of this row tile's previous step
                // (n_mine tiles back, so every group but possibly the latest) have completed
                // before its rows are read back (each warp's lane 0 issued some of them)
                if (e.lane == 0) {
                    if (e.n_mine == 1)
                        tc::bulk_wait();
                    else
                        tc::bulk_wait_all_but_last();
                }
                __syncwarp();
                tc::bar_sync(3, E * 32);
            }
#pragma unroll
            for (int cg = 0; cg < UE / NG; ++cg) {
                const int u = u0 + cg * NG;
                if (row_ok && u < H) {
                    ld_f<NG>(a.hist_c + ((size_t)src * B + b) * H + u, cr + cg * NG);
                    if (!is_new) ld_h<NG>(a.hr + ((size_t)s_next * B + b) * H + u, hc + cg * NG / 2);
                }
            }
            if (pf_early) prefetch_next();
            if (e.lane == 0) tc::bulk_wait_read();  // the previous tile's stores read the staging tiles
            const bool ok = tc::mbar_wait(&e.c.tfull[acc], (k >> 1) & 1, e.limit, e.c.abort);
            if (!ok) ws_abort(e.c, a.err);
            __syncwarp();
            if (tc::bar_any(1, E * 32, !ok || *e.c.abort)) break;
            tc::tc_fence_after();
            // the four gates' pre-activations: all UE units at once, or (more than 16
            // units a thread) group by group, which bounds the registers they take
            constexpr bool kByGroup = UE > 16;
            constexpr int ZW = kByGroup ? NG : UE;
            uint32_t zr[4][ZW];
            if constexpr (!kByGroup) {
#pragma unroll
                for (int g = 0; g < 4; ++g) tmem_cols<UE>(taddr + g * U + e.part * UE, zr[g]);
                tc::tmem_wait_ld();
                tc::tc_fence_before();
                __syncwarp();
                if (e.lane == 0) tc::mbar_arrive(&e.c.tempty[acc]);
            }
#pragma unroll
            for (int cg = 0; cg < UE / NG; ++cg) {
                const int u = u0 + cg * NG;
                if constexpr (kByGroup) {
#pragma unroll
                    for (int g = 0; g < 4; ++g) tmem_cols<NG>(taddr + g * U + e.part * UE + cg * NG, zr[g]);
                    tc::tmem_wait_ld();
                    if (cg == UE / NG - 1) {
                        tc::tc_fence_before();
                        __syncwarp();
                        if (e.lane == 0) tc::mbar_arrive(&e.c.tempty[acc]);
                    }
                }
                if (!(row_ok && u < H)) continue;
                float cn[NG], hn[NG], gv[4][NG];
#pragma unroll
                for (int i = 0; i < NG; ++i) {
                    const int j = cg * NG + i, jb = e.part * UE + j, jz = kByGroup ? i : j;
                    const float ig = sigm(__uint_as_float(zr[0][jz]) + s_bias[jb]);
                    const float fg = sigm(__uint_as_float(zr[1][jz]) + s_bias[U + jb]);
                    const float gg = tanh_hw(__uint_as_float(zr[2][jz]) + s_bias[2 * U + jb]);
                    const float og = sigm(__uint_as_float(zr[3][jz]) + s_bias[3 * U + jb]);
                    cn[i] = fmaf(fg, cr[j], ig * gg);
                    hn[i] = og * tanh_hw(cn[i]);
                    gv[0][i] = ig; gv[1][i] = fg; gv[2][i] = gg; gv[3][i] = og;
                }
                // history row t + 1, the h operand of step t + 1 (h' when step t pushed,
                // else the older top), the activated gates (fp16) for the backward
                const size_t w = ((size_t)(t + 1) * B + b) * H + u;
                const uint32_t srow = (uint32_t)(e.q * 32 + e.lane);  // staging row
                uint32_t hb[NG / 2];
                pack_bf16<NG>(hn, hb);
                st_h<NG>(a.hr + w, is_new ? hb : hc + cg * NG / 2);
                // h' and c' into their staging tiles
                const uint32_t htile = e.c.stg + 8u * U * kRows + (uint32_t)(e.part * kRows * UE * 2);
                const uint32_t ctile = e.c.stg + 10u * U * kRows + (uint32_t)(e.part * kRows * UE * 4);
#pragma unroll
                for (int i = 0; i < NG / 8; ++i)
                    tc::st_shared_v4(htile + stg_swz<UE * 2>(srow, cg * NG / 8 + i), hb + 4 * i);
#pragma unroll
                for (int i = 0; i < NG / 4; ++i)
                    tc::st_shared_v4(ctile + stg_swz<UE * 4>(srow, cg * NG / 4 + i),
                                     reinterpret_cast<const uint32_t *>(cn) + 4 * i);
                // gates into the staging tile [gate][part][row][UE units]; a tensor store
                // writes them out after the tile (nothing reads them before the backward)
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    uint32_t gw[NG / 2];
                    pack_f16<NG>(gv[g], gw);
                    const uint32_t tile = e.c.stg + (uint32_t)((g * EP + e.part) * kRows * UE * 2);
#pragma unroll
                    for (int i = 0; i < NG / 8; ++i)
                        tc::st_shared_v4(tile + stg_swz<UE * 2>(srow, cg * NG / 8 + i), gw + 4 * i);
                }
            }
        } else if constexpr (kRows4) {
            // Four lanes per row. The accumulator comes out of tensor memory one row per lane
            // (lane = row); each row's 32 values go through a shared-memory tile so that in
            // round j lane l takes row 8 j + l / 4 of the warp's 32, units 8 (l % 4) .. + 7.
            // Every global access of a round then covers eight rows with four lanes on each
            // row's 128-byte line, a quarter of the L1 wavefronts of one row per lane. The
            // history indices of a round's row come from the lane that loaded them.
            const uint32_t xb = e.c.stg + (uint32_t)e.q * 4096u;  // this warp's 32 rows x 128 B
            const int sub = e.lane & 3, us = u0 + 8 * sub;
            float dr[4][8];
            const bool ok = tc::mbar_wait(&e.c.tfull[acc], (k >> 1) & 1, e.limit, e.c.abort);
            if (!ok) ws_abort(e.c, a.err);
            __syncwarp();
            if (tc::bar_any(1, E * 32, !ok || *e.c.abort)) break;
            tc::tc_fence_after();
            {
                uint32_t v[UE];
                tmem_cols<UE>(taddr, v);
                tc::tmem_wait_ld();
                tc::tc_fence_before();
                __syncwarp();
                if (e.lane == 0) tc::mbar_arrive(&e.c.tempty[acc]);
                // row = lane, 16-byte piece i at piece i ^ (row mod 8): conflict-free both ways
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    tc::st_shared_v4(xb + (uint32_t)e.lane * 128u + (uint32_t)((i ^ (e.lane & 7)) * 16), v + 4 * i);
            }
            __syncwarp();
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int rr = 8 * j + (e.lane >> 2);
                r_src[j] = __shfl_sync(0xffffffffu, cur0, rr);
                r_s1[j] = __shfl_sync(0xffffffffu, cur1, rr);
                r_ok[j] = rt * kRows + e.q * 32 + rr < B && us < H;
                uint32_t w[8];
                ld_shared_v4(xb + (uint32_t)rr * 128u + (uint32_t)(((2 * sub) ^ (rr & 7)) * 16), w);
                ld_shared_v4(xb + (uint32_t)rr * 128u + (uint32_t)(((2 * sub + 1) ^ (rr & 7)) * 16), w + 4);
#pragma unroll
                for (int i = 0; i < 8; ++i) dr[j][i] = __uint_as_float(w[i]);
            }
            // two rounds' operands in flight at a time
#pragma unroll
            for (int jp = 0; jp < 4; jp += 2) {
                float dh_src[2][8], dh_t[2][8], dc_t[2][8], cn[2][8], cr[2][8], dc_rd[2][8];
                uint32_t gq[2][4][4];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = jp + h;
                    if (!r_ok[j]) continue;
                    const int bj = rt * kRows + e.q * 32 + 8 * j + (e.lane >> 2);
                    ld_f<8>(a.dhist_h + ((size_t)r_src[j] * B + bj) * H + us, dh_src[h]);
                    if (t >= 1) {
                        const size_t wr = ((size_t)t * B + bj) * H + us, rd = ((size_t)r_s1[j] * B + bj) * H + us;
                        ld_f<8>(a.dhist_h + wr, dh_t[h]);
                        ld_f<8>(a.dhist_c + wr, dc_t[h]);
                        ld_f<8>(a.hist_c + wr, cn[h]);
                        ld_f<8>(a.hist_c + rd, cr[h]);
                        ld_f<8>(a.dhist_c + rd, dc_rd[h]);
                        const __half *gt = a.gates + ((size_t)(t - 1) * B + bj) * 4 * H + us;
#pragma unroll
                        for (int g = 0; g < 4; ++g) ld_v4(gt + (size_t)g * H, gq[h][g]);
                    }
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int j = jp + h;
                    if (!r_ok[j]) continue;
                    float v[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) v[i] = dh_src[h][i] + dr[j][i];
#pragma unroll
                    for (int i = 0; i < 8; ++i) dfh[8 * j + i] = v[i];
                    if (t >= 1) {
                        const int bj = rt * kRows + e.q * 32 + 8 * j + (e.lane >> 2);
                        float ig[8], fg[8], gg[8], og[8], d[4][8];
                        unpack_f16<8>(gq[h][0], ig);
                        unpack_f16<8>(gq[h][1], fg);
                        unpack_f16<8>(gq[h][2], gg);
                        unpack_f16<8>(gq[h][3], og);
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float dh = r_src[j] == t ? v[i] : dh_t[h][i];  // the state read at t is row t
                            const float tcn = tanh_hw(cn[h][i]);
                            const float dc = dc_t[h][i] + dh * og[i] * (1.0f - tcn * tcn);
                            d[0][i] = dc * gg[i] * ig[i] * (1.0f - ig[i]);
                            d[1][i] = dc * cr[h][i] * fg[i] * (1.0f - fg[i]);
                            d[2][i] = dc * ig[i] * (1.0f - gg[i] * gg[i]);
                            d[3][i] = dh * tcn * og[i] * (1.0f - og[i]);
                            dfc[8 * j + i] = dc_rd[h][i] + dc * fg[i];
                        }
                        __nv_bfloat16 *dg = a.dG + ((size_t)(t - 1) * B + bj) * 4 * H + us;
#pragma unroll
                        for (int g = 0; g < 4; ++g) {
                            uint32_t w[4];
                            pack_bf16<8>(d[g], w);
                            st_v4(dg + (size_t)g * H, w);
                        }
                    }
                }
            }
        } else {
            // Epilogue operands: the gradient history of this thread's units is written only
            // by this thread (or zeroed before the launch); gates and cell states come from
            // the forward. With one access group per thread they are loaded before the
            // accumulator wait; with several, group by group (their lines are already on
            // their way to L2), which bounds the registers they hold.
            constexpr int NGRP = UE / NG;
            constexpr bool kEarly = UE <= 16;
            constexpr int NO = kEarly ? UE : NG;  // units whose operands are held at once
            const int src = cur0, s1 = cur1;
            float dh_src[NO], dh_t[NO], dc_t[NO], cn[NO], cr[NO], dc_rd[NO];
            uint32_t gq[4][NO / 2];
            // operands of units u .. u + NG - 1 into slot j (units j * NG ..) of the arrays
            auto load_ops = [&](int u, int j) {
                ld_f<NG>(a.dhist_h + ((size_t)src * B + b) * H + u, dh_src + j * NG);
                if (t >= 1) {
                    const size_t wr = ((size_t)t * B + b) * H + u, rd = ((size_t)s1 * B + b) * H + u;
                    ld_f<NG>(a.dhist_h + wr, dh_t + j * NG);
                    ld_f<NG>(a.dhist_c + wr, dc_t + j * NG);
                    ld_f<NG>(a.hist_c + wr, cn + j * NG);
                    ld_f<NG>(a.hist_c + rd, cr + j * NG);
                    ld_f<NG>(a.dhist_c + rd, dc_rd + j * NG);
                    const __half *gt = a.gates + ((size_t)(t - 1) * B + b) * 4 * H + u;
#pragma unroll
                    for (int g = 0; g < 4; ++g) ld_h<NG>(gt + (size_t)g * H, gq[g] + j * NG / 2);
                }
            };
            if (kEarly) {
                prefetch_next();
#pragma unroll
                for (int cg = 0; cg < NGRP; ++cg)
                    if (row_ok && u0 + cg * NG < H) load_ops(u0 + cg * NG, cg);
            }
            const bool ok = tc::mbar_wait(&e.c.tfull[acc], (k >> 1) & 1, e.limit, e.c.abort);
            if (!ok) ws_abort(e.c, a.err);
            __syncwarp();
            if (tc::bar_any(1, E * 32, !ok || *e.c.abort)) break;
            tc::tc_fence_after();
            float dsum[KS > 1 ? UE : 1];
            if constexpr (KS > 1) {
                // this lane's whole partial row, then the sum of the parts for its units
                uint32_t pr[U];
                tmem_cols<U>(taddr, pr);
                tc::tmem_wait_ld();
                tc::tc_fence_before();
                __syncwarp();
                if (e.lane == 0) tc::mbar_arrive(&e.c.tempty[acc]);
#pragma unroll
                for (int i = 0; i < UE; ++i) dsum[i] = 0.0f;
                if (p.cl > 1) {
                    // the parts form a cluster: this row's units of part j go straight into
                    // CTA j's exchange tile by asynchronous stores that count their bytes on
                    // its barrier; this tile's phase completes once the other parts' bytes
                    // landed and thread 0 arrived with their count (one row tile per CTA: a
                    // part stores a tile's partials only after every CTA of the row tile
                    // released the step before, so after this CTA read the previous ones)
                    constexpr int G4 = UE / 4;
                    const uint32_t r16 = (uint32_t)(e.q * 32 + e.lane) * 16u;
                    if (e.tid == 0) tc::mbar_arrive_expect_tx(e.c.rbar, (uint32_t)(KS - 1) * kRows * UE * 4);
#pragma unroll
                    for (int j = 0; j < KS; ++j) {
                        if (j == e.kp) continue;
                        const uint32_t dst = tc::mapa(e.c.xch, (uint32_t)j) + (uint32_t)(e.kp * G4) * (kRows * 16u) + r16;
                        const uint32_t bar = tc::mapa(tc::smem_u32(e.c.rbar), (uint32_t)j);
#pragma unroll
                        for (int g = 0; g < G4; ++g) tc::st_async_v4(dst + (uint32_t)g * (kRows * 16u), pr + j * UE + 4 * g, bar);
                    }
                    const bool ok2 = tc::mbar_wait_cluster(e.c.rbar, (uint32_t)(k & 1), e.limit, e.c.abort);
                    if (!ok2) ws_abort(e.c, a.err);
                    __syncwarp();
                    if (tc::bar_any(1, E * 32, !ok2 || *e.c.abort)) break;
                    // the sum in part order, as below
#pragma unroll
                    for (int j = 0; j < KS; ++j) {
#pragma unroll
                        for (int g = 0; g < G4; ++g) {
                            uint32_t w[4];
                            if (j == e.kp) {
#pragma unroll
                                for (int i = 0; i < 4; ++i) w[i] = pr[j * UE + 4 * g + i];
                            } else {
                                ld_shared_v4(e.c.xch + (uint32_t)(j * G4 + g) * (kRows * 16u) + r16, w);
                            }
#pragma unroll
                            for (int i = 0; i < 4; ++i) dsum[4 * g + i] += __uint_as_float(w[i]);
                        }
                    }
                } else {
                    // the whole partial row of this lane to the L2 scratch, counted, then the
                    // parts of this CTA's units read back once every part counted
                    const size_t grp = (size_t)rt * p.n_ct + e.ct;
                    float *prow = p.part + ((grp * KS + e.kp) * kRows + e.q * 32 + e.lane) * U;
#pragma unroll
                    for (int i = 0; i < U / 8; ++i) st_v8(prow + 8 * i, pr + 8 * i);
                    __syncwarp();
                    tc::bar_sync(2, E * 32);
                    bool ok2 = true;
                    if (e.tid == 0) {
                        tc::red_release_gpu_add(p.pcnt + grp, 1);
                        ok2 = spin_until(p.pcnt + grp, KS * (ks + 1), e.limit, e.c.abort, a.err);
                        if (!ok2) ws_abort(e.c, a.err);
                    }
                    __syncwarp();
                    if (tc::bar_any(1, E * 32, !ok2 || *e.c.abort)) break;
#pragma unroll
                    for (int j = 0; j < KS; ++j) {
                        float v[UE];
                        ld_f<UE>(p.part + ((grp * KS + j) * kRows + e.q * 32 + e.lane) * U + e.kp * (U / KS), v);
#pragma unroll
                        for (int i = 0; i < UE; ++i) dsum[i] += v[i];
                    }
                }
            }
#pragma unroll
            for (int cg = 0; cg < NGRP; ++cg) {
                const int u = u0 + cg * NG;
                const int j = kEarly ? cg : 0;  // operand slot of this group
                uint32_t dr[NG];
                if constexpr (KS > 1) {
#pragma unroll
                    for (int i = 0; i < NG; ++i) dr[i] = __float_as_uint(dsum[cg * NG + i]);
                } else {
                    tmem_cols<NG>(taddr + e.part * UE + cg * NG, dr);
                    tc::tmem_wait_ld();
                    if (cg == NGRP - 1) {
                        tc::tc_fence_before();
                        __syncwarp();
                        if (e.lane == 0) tc::mbar_arrive(&e.c.tempty[acc]);
                    }
                }
                const bool mine = row_ok && u < H;
                if (!kEarly && mine) load_ops(u, 0);
                if (!mine) continue;
                float v[NG];
#pragma unroll
                for (int i = 0; i < NG; ++i) v[i] = dh_src[j * NG + i] + __uint_as_float(dr[i]);
                if constexpr (kDeferDhist) {
#pragma unroll
                    for (int i = 0; i < NG; ++i) dfh[cg * NG + i] = v[i];
                } else {
                    st_f<NG>(a.dhist_h + ((size_t)src * B + b) * H + u, v);
                }
                if (t >= 1) {
                    float ig[NG], fg[NG], gg[NG], og[NG], d[4][NG], dcr[NG];
                    unpack_f16<NG>(gq[0] + j * NG / 2, ig);
                    unpack_f16<NG>(gq[1] + j * NG / 2, fg);
                    unpack_f16<NG>(gq[2] + j * NG / 2, gg);
                    unpack_f16<NG>(gq[3] + j * NG / 2, og);
#pragma unroll
                    for (int i = 0; i < NG; ++i) {
                        const int q = j * NG + i;
                        const float dh = src == t ? v[i] : dh_t[q];  // the state read at t is row t
                        const float tcn = tanh_hw(cn[q]);
                        const float dc = dc_t[q] + dh * og[i] * (1.0f - tcn * tcn);
                        d[0][i] = dc * gg[i] * ig[i] * (1.0f - ig[i]);
                        d[1][i] = dc * cr[q] * fg[i] * (1.0f - fg[i]);
                        d[2][i] = dc * ig[i] * (1.0f - gg[i] * gg[i]);
                        d[3][i] = dh * tcn * og[i] * (1.0f - og[i]);
                        dcr[i] = dc_rd[q] + dc * fg[i];
                    }
                    __nv_bfloat16 *dg = a.dG + ((size_t)(t - 1) * B + b) * 4 * H + u;
#pragma unroll
                    for (int g = 0; g < 4; ++g) {
                        uint32_t w[NG / 2];
                        pack_bf16<NG>(d[g], w);
                        st_h<NG>(dg + (size_t)g * H, w);
                    }
                    if constexpr (kDeferDhist) {
#pragma unroll
                        for (int i = 0; i < NG; ++i) dfc[cg * NG + i] = dcr[i];
                    } else {
                        st_f<NG>(a.dhist_c + ((size_t)s1 * B + b) * H + u, dcr);
                    }
                }
            }
            d_src = src;
            d_s1 = s1;
        }
        if (kFwd ? !pf_early : kLatePfBwd) prefetch_next();
        // the next step reads these rows by TMA: generic writes -> async proxy; then, with
        // the release warp, which releases the step for this row tile while this tile's
        // remaining stores go out and the next tile starts
        tc::fence_proxy_async_global();
        if constexpr (kFwd) tc::fence_proxy_async();  // staging-tile writes -> the tensor store
        __syncwarp();
        if (rel_warp<U, EP, kFwd, KS>(p)) {
            tc::bar_sync(kRelBar, (E + 1) * 32);
        } else {
            tc::bar_sync(2, E * 32);
            if (e.tid == 0) tc::red_release_gpu_add(p.cnt + rt * p.cs, 1);
        }
        if constexpr (kRows4) {
            const int sub = e.lane & 3, us = u0 + 8 * sub;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (!r_ok[j]) continue;
                const int bj = rt * kRows + e.q * 32 + 8 * j + (e.lane >> 2);
                st_f<8>(a.dhist_h + ((size_t)r_src[j] * B + bj) * H + us, dfh + 8 * j);
                if (t >= 1) st_f<8>(a.dhist_c + ((size_t)r_s1[j] * B + bj) * H + us, dfc + 8 * j);
            }
        } else if constexpr (kDeferDhist) {
            if (row_ok) {
#pragma unroll
                for (int cg = 0; cg < UE / NG; ++cg) {
                    const int u = u0 + cg * NG;
                    if (u >= H) continue;
                    st_f<NG>(a.dhist_h + ((size_t)d_src * B + b) * H + u, dfh + cg * NG);
                    if (t >= 1) st_f<NG>(a.dhist_c + ((size_t)d_s1 * B + b) * H + u, dfc + cg * NG);
                }
            }
        }
        if constexpr (kFwd) {
            // the tile's 6 EP tensor stores (4 EP gate blocks, EP h' and EP c' blocks), issued
            // by lane 0 of the epilogue warps, store w, w + E, ... each
            if (e.lane == 0) {
                const int w = e.part * 4 + e.q;
                for (int st = w; st < 6 * EP; st += E) {
                    if (st < 4 * EP) {
                        const int g = st / EP, q = st % EP;
                        tc::tma_store_4d(tm_gates, e.c.stg + (uint32_t)((g * EP + q) * kRows * UE * 2),
                                         e.ct * U + q * UE, g, rt * kRows, t);
                    } else if (st < 5 * EP) {
                        const int q = st - 4 * EP;
                        tc::tma_store_3d(tm_hh, e.c.stg + 8u * U * kRows + (uint32_t)(q * kRows * UE * 2),
                                         e.ct * U + q * UE, rt * kRows, t + 1);
                    } else {
                        const int q = st - 5 * EP;
                        tc::tma_store_3d(tm_hc, e.c.stg + 10u * U * kRows + (uint32_t)(q * kRows * UE * 4),
                                         e.ct * U + q * UE, rt * kRows, t + 1);
                    }
                }
                tc::bulk_commit();
            }
        }
        cur0 = nx0;
        cur1 = nx1;
    }
    // the release warp's last barrier, after every tile (or after an abort, at the tile the
    // epilogue left): the tiles completed, k, tell it that this one releases nothing
    if (rel_warp<U, EP, kFwd, KS>(p)) {
        if (e.tid == 0) *e.c.rel_end = k;
        tc::bar_sync(kRelBar, (E + 1) * 32);
    }
    if constexpr (kFwd)
        if (e.lane == 0) tc::bulk_wait();  // the history stores completed before the CTA exits
}

// ------------------------------------------------------------------ input gradient
// Backward only. The CTAs past the step chain compute dx = dG W_x^T (the input part of the
// gate-gradient contraction, Sec. 5) on SMs the chain leaves idle. The [T B][4H] gate
// gradient is cut into 128-row tiles, taken from the last row down so that each tile
// trails the chain step that completed it; this CTA takes every n_dx-th (tile, 256-column
// slice of dx) pair. Before loading a tile whose earliest row belongs to step t_lo, the
// producer waits until every row tile of the chain has completed T - 1 - t_lo steps
// (chain step t writes the gate gradient of step t - 1, so the rows of t_lo and later are
// then final), then streams the 4H / 64 contraction chunks with the matching 256-row
// slices of W_x through an S-stage ring. Accumulators alternate between the two 256-column halves of tensor memory; the
// epilogue warps store their rows of the finished one while the next tile is multiplied.
// The role is inlined into the kernel: compiled as a called function, its 32-byte row
// stores wrote only their first word (found with a NaN-filled output).
constexpr int kDxN = 256;

template <int EP>
__device__ __forceinline__ void dx_role(const CUtensorMap *tm_g, const WsArgs &p, uint8_t *smem_raw, int per_step)
{
    constexpr int E = 4 * EP;
    constexpr int CPT = kDxN / EP;  // dx columns per epilogue thread
    constexpr uint32_t kWChunk = kDxN * 128;
    const StepArgs &a = p.s;
    const int T = a.T, B = a.B, I = a.I, KC = a.KC, S = p.dx_S;
    const size_t R = (size_t)T * B;
    const int n_rows = (int)((R + kRows - 1) / kRows);
    const int n_items = n_rows * p.nxt;
    const int did = (int)blockIdx.x - p.n_chain;
    const int n_mine = did < n_items ? (n_items - did + p.n_dx - 1) / p.n_dx : 0;
    const long long limit = a.limit;
    const WCtl c = wcarve(smem_raw, S, 1, kDxN, KC, 0, 0u, 0u);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(&c.full[s], 1);
            tc::mbar_init(&c.empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&c.tfull[i], 1);
            tc::mbar_init(&c.tempty[i], E);
        }
        tc::mbar_init(c.done, 1);
        *c.n_issued = 0;
        *c.n_consumed = 0;
        *c.abort = 0;
        tc::fence_mbar_init();
    }
    if (warp == E) tc::tmem_alloc(c.tmem_slot, 2 * kDxN);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *c.tmem_slot;
    auto item = [&](int j, int &row0, int &xt) {
        const int i = did + j * p.n_dx;
        row0 = (n_rows - 1 - i / p.nxt) * kRows;
        xt = i % p.nxt;
    };

    if (warp == E) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t g = 0;
            for (int j = 0; j < n_mine && !*c.abort; ++j) {
                int row0, xt;
                item(j, row0, xt);
                // the row tiles holding the tile's rows: instances b0 .. of step t_lo, and
                // (B >= 128) at most instances 0 .. 127 of step t_lo + 1; polled slowly, as
                // the chain's own hand-offs use the same counters
                const int t_lo = row0 / B, b0 = row0 - t_lo * B, b1 = min(B - 1, b0 + kRows - 1);
                bool ok = true;
                for (int rt = b0 / kRows; rt <= b1 / kRows && ok; ++rt)
                    ok = spin_until(p.cnt + rt * p.cs, per_step * (T - 1 - t_lo), limit, c.abort, a.err, 1000);
                if (ok && b0 + kRows > B && t_lo + 1 < T)
                    ok = spin_until(p.cnt, per_step * (T - 2 - t_lo), limit, c.abort, a.err, 1000);
                if (!ok) {
                    ws_abort(c, a.err);
                    break;
                }
                tc::fence_proxy_async_global();
                const uint8_t *wt = p.wdx + (size_t)xt * KC * kWChunk;
                bool bad = false;
                for (int kc = 0; kc < KC; ++kc) {
                    const int s = (int)(g % S);
                    if (g >= (uint32_t)S && !tc::mbar_wait(&c.empty[s], (g / S - 1) & 1, limit, c.abort)) {
                        ws_abort(c, a.err);
                        bad = true;
                        break;
                    }
                    const uint32_t st = c.ring0 + s * c.stage;
                    tc::mbar_arrive_expect_tx(&c.full[s], kAStage + kWChunk);
                    tc::tma_load_2d(st, tm_g, kc * kChunk, row0, &c.full[s]);
                    tc::bulk_g2s(st + kAStage, wt + (size_t)kc * kWChunk, kWChunk, &c.full[s]);
                    ++g;
                }
                if (bad) break;
            }
            *c.n_issued = (int)g;
        }
        __syncwarp();
    } else if (warp == E + 1) {
        // ------------------------------------------------------------ MMA issue
        if (lane == 0) {
            uint32_t g = 0;
            for (int j = 0; j < n_mine && !*c.abort; ++j) {
                const int acc = j & 1;
                if (j >= 2 && !tc::mbar_wait(&c.tempty[acc], ((j >> 1) - 1) & 1, limit, c.abort)) {
                    ws_abort(c, a.err);
                    break;
                }
                tc::tc_fence_after();
                const uint32_t d = tmem + acc * kDxN;
                bool bad = false;
                for (int kc = 0; kc < KC; ++kc) {
                    const int s = (int)(g % S);
                    if (!tc::mbar_wait(&c.full[s], (g / S) & 1, limit, c.abort)) {
                        ws_abort(c, a.err);
                        bad = true;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t st = c.ring0 + s * c.stage;
                    issue_group<kDxN, 1>(d, st, st + kAStage, 1, kc == 0);
                    tc::mma_commit(&c.empty[s]);
                    ++g;
                }
                if (bad) break;
                tc::mma_commit(&c.tfull[acc]);
            }
            *c.n_consumed = (int)g;
            tc::mma_commit(c.done);
        }
        __syncwarp();
    } else if (warp < E) {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3, part = warp >> 2;
        for (int j = 0; j < n_mine; ++j) {
            int row0, xt;
            item(j, row0, xt);
            const int acc = j & 1;
            const bool ok = tc::mbar_wait(&c.tfull[acc], (j >> 1) & 1, limit, c.abort);
            if (!ok) {
                ws_abort(c, a.err);
                break;
            }
            tc::tc_fence_after();
            const size_t row = (size_t)row0 + q * 32 + lane;
            const uint32_t taddr = tmem + acc * kDxN + ((uint32_t)(q * 32) << 16) + part * CPT;
            // the dx row of this accumulator row: the same row, or (push-only mode) the
            // real step of this virtual row's push; rows past an instance's pushes have none
            bool out = row < R;
            size_t orow = row;
            if (out && p.dx_xidx) {
                const int tr = p.dx_xidx[row];
                out = tr >= 0;
                orow = (size_t)tr * B + row % B;
            }
            float *drow = p.dx + orow * I;
#pragma unroll 1
            for (int cg = 0; cg < CPT / 16; ++cg) {
                uint32_t v[16];
                tmem_cols<16>(taddr + cg * 16, v);
                tc::tmem_wait_ld();
                const int col = xt * kDxN + part * CPT + cg * 16;
                if (out) {
#pragma unroll
                    for (int h = 0; h < 2; ++h)
                        if (col + 8 * h < I) {  // I is a multiple of 8
                            if (p.dx_v8)
                                st_v8(drow + col + 8 * h, v + 8 * h);
                            else {
                                st_v4(drow + col + 8 * h, v + 8 * h);
                                st_v4(drow + col + 8 * h + 4, v + 8 * h + 4);
                            }
                        }
                }
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(&c.tempty[acc]);
        }
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == E && lane == 0)
        for (int g = *c.n_consumed; g < *c.n_issued; ++g)
            tc::mbar_wait(&c.full[g % S], (uint32_t)(g / S) & 1, kDrainLimit, nullptr);
    if (warp == E + 1 && lane == 0) tc::mbar_wait(c.done, 0, kDrainLimit, nullptr);
    tc::tc_fence_before();
    __syncthreads();
    if (warp == E) tc::tmem_dealloc(tmem, 2 * kDxN);
}

// ------------------------------------------------------------------ the kernel
// kFwd: forward (tm_a = x_t tiles for chunks < kcx, tm_b = hr[t] tiles after them);
// else backward (tm_b = dG_t tiles, kcx = 0: every chunk depends on the step before).
// KS > 1 (backward): the KS CTAs blockIdx = (slot, ct, kp) split the contraction; part kp
// takes chunks [KC kp / KS, KC (kp + 1) / KS) and keeps only that slice of the weight tile.
template <int U, int EP, int G, bool kFwd, int KS>
__global__ void __launch_bounds__(32 * (4 * EP + 3), 1)
step_ws(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
        const __grid_constant__ CUtensorMap tm_gates, const __grid_constant__ CUtensorMap tm_hh,
        const __grid_constant__ CUtensorMap tm_hc, WsArgs p)
{
    constexpr int NB = kFwd ? 4 * U : U;  // accumulator columns
    constexpr int E = 4 * EP;             // epilogue warps
    constexpr int UE = U / KS / EP;       // units each epilogue thread finishes
    constexpr uint32_t kCols = TmemCols<NB>::value;
    constexpr uint32_t bchunk = NB * 128;
    static_assert(UE % 8 == 0, "epilogue works on groups of 8 units");
    const StepArgs &a = p.s;
    extern __shared__ uint8_t smem_raw[];
    __shared__ float s_bias[kFwd ? 4 * U : 4];
    if constexpr (!kFwd)
        if ((int)blockIdx.x >= p.n_chain) {
            dx_role<EP>(&tm_b, p, smem_raw, p.n_ct * KS);
            return;
        }
    const int S = a.S, KC = a.KC, split = a.kcx, T = a.T, B = a.B, H = a.H;
    const int kp = (int)(blockIdx.x % KS), cidx = (int)(blockIdx.x / KS);
    const int k0 = KC * kp / KS, k1 = KC * (kp + 1) / KS;  // this CTA's contraction chunks
    const int dep_c = split > k0 ? split : k0;            // first chunk that needs step t - 1
    // the parts trade partials in the cluster's shared memory; a launch whose clusters are not
    // the KS parts of a column tile (blockIdx.x % KS is the rank only then) takes the L2
    // exchange instead, so no CTA ever addresses a peer that is not there
    const bool xcl = KS > 1 && p.cl > 1 && tc::cluster_size() == (uint32_t)KS;
    const WCtl c = wcarve(smem_raw, S, G, NB, (KC + KS - 1) / KS, p.w_res, ws_stg_bytes(kFwd, U),
                          xcl ? ws_xch_bytes(U) : 0u);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int ct = cidx % p.n_ct, slot = cidx / p.n_ct;
    const int n_mine = slot < p.n_rt ? (p.n_rt - slot + p.n_slot - 1) / p.n_slot : 0;
    const int n_tiles = T * n_mine;
    const long long limit = a.limit;
    if (kFwd)
        for (int i = tid; i < 4 * U; i += blockDim.x) {
            const int g = i / U, u = ct * U + i % U;
            s_bias[i] = u < H ? a.bias[g * H + u] : 0.0f;
        }
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(&c.full[s], 1);
            tc::mbar_init(&c.empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(&c.tfull[i], 1);
            tc::mbar_init(&c.tempty[i], E);
        }
        tc::mbar_init(c.wbar, 1);
        tc::mbar_init(c.done, 1);
        // one arrival a tile (with the bytes the other parts store asynchronously)
        tc::mbar_init(c.rbar, 1);
        *c.n_issued = 0;
        *c.n_consumed = 0;
        *c.abort = 0;
        *c.rel_end = 0x7fffffff;
        tc::fence_mbar_init();
    }
    if (warp == E) tc::tmem_alloc(c.tmem_slot, 2 * kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (xcl) tc::cluster_sync();  // the other parts' barriers are initialised before any arrival
    const uint32_t tmem = *c.tmem_slot;
    const uint8_t *wtile = a.wpack + (size_t)ct * KC * bchunk;

    if (warp == E) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            if (p.w_res) {
                tc::mbar_arrive_expect_tx(c.wbar, (k1 - k0) * bchunk);
                tc::bulk_g2s(c.w0, wtile + (size_t)k0 * bchunk, (k1 - k0) * bchunk, c.wbar);
            }
            uint32_t g = 0;
            for (int k = 0; k < n_tiles && !*c.abort; ++k) {
                const int ks = k / n_mine, rt = slot + (k % n_mine) * p.n_slot;
                const int t = kFwd ? ks : T - 1 - ks;
                const int row = t * B + rt * kRows;
                int armed = 0;  // next groups whose stage is armed and weight chunks issued
                bool bad = false;
                for (int c0 = k0; c0 < k1;) {
                    const int c1 = group_end(c0, G, split, k1);
                    if (c0 == dep_c && ks > 0) {
                        // backward: streamed weight chunks do not depend on the step before:
                        // the first groups whose stages are already free are armed and get
                        // their weight copies before the wait, so that only the dG rows
                        // remain to load once it ends (large backward -1.7 %; the forward,
                        // whose x part fills the ring just before, measured slower)
                        if (!kFwd && !p.w_res)
                            for (int d0 = c0; d0 < k1 && armed < S;) {
                                const int d1 = group_end(d0, G, split, k1);
                                const uint32_t gd = g + (uint32_t)armed;
                                const int sd = (int)(gd % S);
                                if (gd >= (uint32_t)S && !tc::mbar_test_wait(&c.empty[sd], (gd / S - 1) & 1)) break;
                                tc::mbar_arrive_expect_tx(&c.full[sd], (d1 - d0) * ((uint32_t)p.a_rows * 128 + bchunk));
                                tc::bulk_g2s(c.ring0 + sd * c.stage + G * kAStage, wtile + (size_t)d0 * bchunk,
                                             (d1 - d0) * bchunk, &c.full[sd]);
                                ++armed;
                                d0 = d1;
                            }
                        // every column tile (and contraction part) of this row tile
                        // finished the step before
                        if (!spin_until(p.cnt + rt * p.cs, p.n_ct * KS * ks, limit, c.abort, a.err)) {
                            ws_abort(c, a.err);
                            bad = true;  // armed stages still get their (unused) rows, so they complete
                        } else {
                            tc::fence_proxy_async_global();
                        }
                    }
                    if (bad && armed == 0) break;
                    const int s = (int)(g % S);
                    const uint32_t st = c.ring0 + s * c.stage;
                    const bool pre = armed > 0;
                    if (pre) {
                        --armed;
                    } else {
                        if (g >= (uint32_t)S && !tc::mbar_wait(&c.empty[s], (g / S - 1) & 1, limit, c.abort)) {
                            ws_abort(c, a.err);
                            bad = true;
                            break;
                        }
                        tc::mbar_arrive_expect_tx(&c.full[s],
                                                  (c1 - c0) * ((uint32_t)p.a_rows * 128 + (p.w_res ? 0u : bchunk)));
                    }
                    for (int cc = c0; cc < c1; ++cc) {
                        const bool first = cc < split;
                        const CUtensorMap *tm = first ? &tm_a : &tm_b;
                        const int col = (first ? cc : cc - split) * kChunk;
                        const uint32_t dst = st + (cc - c0) * kAStage;
                        tc::tma_load_2d(dst, tm, col, row, &c.full[s]);
                    }
                    if (!pre && !p.w_res)
                        tc::bulk_g2s(st + G * kAStage, wtile + (size_t)c0 * bchunk, (c1 - c0) * bchunk, &c.full[s]);
                    ++g;
                    c0 = c1;
                }
                if (bad) break;
            }
            *c.n_issued = (int)g;
        }
        __syncwarp();
    } else if (warp == E + 1) {
        // ------------------------------------------------------------ MMA issue
        if (lane == 0) {
            uint32_t g = 0;
            bool w_ready = !p.w_res;
            for (int k = 0; k < n_tiles && !*c.abort; ++k) {
                const int acc = k & 1;
                if (k >= 2 && !tc::mbar_wait(&c.tempty[acc], ((k >> 1) - 1) & 1, limit, c.abort)) {
                    ws_abort(c, a.err);
                    break;
                }
                if (!w_ready) {
                    if (!tc::mbar_wait(c.wbar, 0, limit, c.abort)) {
                        ws_abort(c, a.err);
                        break;
                    }
                    w_ready = true;
                }
                tc::tc_fence_after();
                const uint32_t d = tmem + acc * kCols;
                bool bad = false;
                for (int c0 = k0; c0 < k1;) {
                    const int c1 = group_end(c0, G, split, k1);
                    const int s = (int)(g % S);
                    if (!tc::mbar_wait(&c.full[s], (g / S) & 1, limit, c.abort)) {
                        ws_abort(c, a.err);
                        bad = true;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t st = c.ring0 + s * c.stage;
                    issue_group<NB, G>(d, st, p.w_res ? c.w0 + (c0 - k0) * bchunk : st + G * kAStage, c1 - c0,
                                       c0 == k0);
                    tc::mma_commit(&c.empty[s]);
                    ++g;
                    c0 = c1;
                }
                if (bad) break;
                tc::mma_commit(&c.tfull[acc]);
            }
            *c.n_consumed = (int)g;
            tc::mma_commit(c.done);  // arrives once every MMA issued above has completed
        }
        __syncwarp();
    } else if (warp == E + 2) {
        // ------------------------------------------------------------ release
        // (only where rel_warp: see kRelBar) once the epilogue warps of tile k have written
        // and fenced its rows (their barrier), count the step done for the tile's row tile,
        // with release semantics. The epilogue ends with one more barrier, before which it
        // records the tiles it completed: that barrier (k == *rel_end) releases nothing and
        // ends this loop, also after an abort
        if (rel_warp<U, EP, kFwd, KS>(p)) {
            for (int k = 0;; ++k) {
                tc::bar_sync(kRelBar, (E + 1) * 32);
                if (k >= *c.rel_end) break;
                if (lane == 0) tc::red_release_gpu_add(p.cnt + (slot + (k % n_mine) * p.n_slot) * p.cs, 1);
                __syncwarp();
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        constexpr int NG = UE % 16 == 0 ? 16 : 8;
        const EpiCtx e{c, tmem, warp & 3, warp >> 2, lane, tid, ct, kp, slot, n_mine, n_tiles, limit};
        if (NG == 16 && p.vec32)
            epilogue_loop<U, EP, NG, kFwd, KS>(a, p, e, s_bias, &tm_gates, &tm_hh, &tm_hc);
        else
            epilogue_loop<U, EP, 8, kFwd, KS>(a, p, e, s_bias, &tm_gates, &tm_hh, &tm_hc);
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == E && lane == 0) {
        // copies still in flight after an abort: stages armed but never consumed
        for (int g = *c.n_consumed; g < *c.n_issued; ++g)
            tc::mbar_wait(&c.full[g % S], (uint32_t)(g / S) & 1, kDrainLimit, nullptr);
        if (p.w_res) tc::mbar_wait(c.wbar, 0, kDrainLimit, nullptr);
    }
    if (warp == E + 1 && lane == 0) tc::mbar_wait(c.done, 0, kDrainLimit, nullptr);
    tc::tc_fence_before();
    __syncthreads();
    if (warp == E) tc::tmem_dealloc(tmem, 2 * kCols);
    // no part leaves while another may still store into its shared memory
    if (xcl) tc::cluster_sync();
}

// ------------------------------------------------------------------ planning
// Measured back-to-back issue cost (cycles) of one M = 128, K = 16 MMA by N, and the
// extra issue stall of one mbarrier wait between MMA runs.
double mma_cycles(int N) { return N <= 16 ? 45 : N <= 32 ? 51 : N <= 64 ? 47 : N <= 128 ? 65 : 128; }
constexpr double kWaitCycles = 300;

struct Variant {
    int U, EP, G, KS;
    const void *fn;
};

template <int U, int EP, int G, bool kFwd, int KS = 1>
Variant variant()
{
    return Variant{U, EP, G, KS, (const void *)step_ws<U, EP, G, kFwd, KS>};
}

const Variant *fwd_variants(int *n)
{
    static const Variant v[] = {variant<8, 1, 4, true>(),  variant<16, 1, 4, true>(), variant<16, 2, 4, true>(),
                                variant<32, 2, 2, true>(), variant<32, 4, 2, true>()};
    *n = 5;
    return v;
}
const Variant *bwd_variants(int *n)
{
    static const Variant v[] = {variant<16, 1, 4, false>(), variant<16, 2, 4, false>(), variant<32, 2, 4, false>(),
                                variant<32, 4, 4, false>(), variant<64, 2, 2, false>(), variant<64, 1, 2, false, 4>(),
                                variant<64, 1, 4, false, 4>(), variant<64, 2, 4, false>(), variant<32, 1, 4, false>()};
    *n = 9;
    return v;
}

// Largest residency (CTAs per SM) that leaves every CTA its two accumulators in tensor
// memory (512 columns per SM); shared memory is padded to enforce it.
uint32_t pad_for_tmem(const void *fn, int threads, uint32_t smem, uint32_t kcols2)
{
    const int max_res = std::max(1, (int)(512 / kcols2));
    for (; smem <= kSmemCap; smem += 4096) {
        int r = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, fn, threads, smem) != cudaSuccess) {
            cudaGetLastError();
            return 0;
        }
        if (r <= max_res) return smem;
    }
    return kSmemCap;
}

// Co-resident thread-block clusters of cl CTAs at this footprint (0 on any error).
int max_clusters(const void *fn, int threads, uint32_t smem, int cl)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cl);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = cl;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

// Plans one variant: the weight tile resident or streamed, a two-stage ring. The grid is
// sized from the number of co-resident CTAs of that footprint. Cost = row-tile rounds per
// step x per-tile time (constants fitted to GB300 measurements); ties go to plans within
// 208 KB of shared memory, then to the resident weight tile.
bool plan_variant(const Variant &v, bool fwd, int KC, int split, int n_rt, int H, int sms, uint32_t cap,
                  PersistPlan *pl, double *cost)
{
    const int NB = fwd ? 4 * v.U : v.U, n_ct = (H + v.U - 1) / v.U;
    const int threads = 32 * (4 * v.EP + 3);  // epilogue warps, producer, MMA issue, release
    const uint32_t kcols2 = 2u * (NB <= 32 ? 32 : NB <= 64 ? 64 : NB <= 128 ? 128 : 256);
    const int KCl = (KC + v.KS - 1) / v.KS;  // chunks of one contraction part
    const int groups = (split + v.G - 1) / v.G + (KCl - split + v.G - 1) / v.G;
    const uint32_t fixed = 1024 + kBarBytes;  // alignment pad and barriers (kSmemCap already leaves static room)
    const int pad = n_ct * v.KS;              // CTAs per row-tile slot
    bool found = false;
    double best = 1e30;
    int best_key = -1;
    if (cudaFuncSetAttribute(v.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemCap) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    for (int wr : {1, 0}) {
        const uint32_t wbytes = wr ? (uint32_t)KCl * NB * 128 : 0u;
        const uint32_t stage = ws_stage_bytes(v.G, NB, wr);
        const uint32_t stg = ws_stg_bytes(fwd, v.U);
        if (fixed + wbytes + stg + 2 * stage > cap) continue;
        // two stages: deeper rings measured slower (their copies compete with the
        // epilogue's loads and stores)
        const int S = 2;
        uint32_t smem = ws_smem_bytes(S, v.G, NB, KCl, wr, stg);
        smem = pad_for_tmem(v.fn, threads, smem, kcols2);
        if (!smem) continue;
        int r = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, v.fn, threads, smem) != cudaSuccess) {
            cudaGetLastError();
            continue;
        }
        const int resident = r * sms;
        if (resident < pad) continue;
        // the fewest slots that give the same number of row-tile rounds per step: every
        // slot then has (about) the same work, and the SMs left over take other work
        const int rounds = (n_rt + std::min(n_rt, resident / pad) - 1) / std::min(n_rt, resident / pad);
        const int sl = (n_rt + rounds - 1) / rounds;
        // a split contraction whose CTAs each keep one row tile: its parts as one
        // thread-block cluster, trading partial sums in shared memory, when the larger
        // footprint and every cluster still fit. Test hook (include/stacklstm.h):
        // STACKLSTM_SPLIT_CLUSTER = 0 keeps the L2 exchange
        int cl = 1;
        if (!fwd && v.KS > 1 && rounds == 1) {
            const char *fc = getenv("STACKLSTM_SPLIT_CLUSTER");
            const uint32_t sx = pad_for_tmem(v.fn, threads, ws_smem_bytes(S, v.G, NB, KCl, wr, stg + ws_xch_bytes(v.U)),
                                             kcols2);
            if ((!fc || atoi(fc) != 0) && sx && sx <= cap &&
                max_clusters(v.fn, threads, sx, v.KS) * v.KS >= pad * sl) {
                cl = v.KS;
                smem = sx;
            }
        }
        // forward, per CTA and step: MMA issue plus the epilogue's ~16 B of stores per
        // (instance, unit) at about 30 B/cycle
        double c = rounds * (KC * 4 * mma_cycles(NB) + groups * kWaitCycles + 128.0 * v.U * 16 / 30);
        if (!fwd) {
            // backward, per CTA and step: the dG operand (and a streamed weight slice)
            // at about 70 B/cycle of TMA ingest against the MMA issue time (about 400
            // cycles per stage wait inside this kernel), then the epilogue's ~48 B per
            // (instance, unit) at about 30 B/cycle of load/store, plus the partial
            // exchange of a split contraction
            const double ingest = (128.0 * KCl * 128 + (wr ? 0.0 : (double)NB * KCl * 128)) / 70;
            const double mma = KCl * 4 * mma_cycles(NB) + groups * 400.0;
            const double xch = v.KS == 1 ? 0.0 : cl > 1 ? 1500.0 : 2.0 * 128 * v.U * 4 / 30 + 3000;
            const double epi = 128.0 * (v.U / v.KS) * 48 / 30 + xch;
            // with two or more row tiles a CTA multiplies one while the epilogue
            // finishes the other (their chains are independent)
            const double mm = std::max(ingest, mma);
            c = rounds > 1 ? rounds * std::max(mm, epi) + std::min(mm, epi) : mm + epi;
        }
        // ties: a plan within 208 KB of shared memory first (beyond it L1 is too small
        // for the epilogue's traffic: the stress forward ran 5% slower with its weight
        // tile resident at 230 KB than streamed at 165 KB), then the resident weight tile
        const int key = (smem <= 208u * 1024) * 10000 + wr * 1000;
        if (c < best * 0.999 || (c <= best * 1.001 && key > best_key)) {
            best = c;
            best_key = key;
            pl->on = 1;
            pl->U = v.U;
            pl->EP = v.EP;
            pl->G = v.G;
            pl->S = S;
            pl->slot = sl;
            pl->w_res = wr;
            pl->cl = cl;
            pl->KS = v.KS;
            pl->n_ct = n_ct;
            pl->smem = smem;
            pl->threads = threads;
            pl->per_sm = r;
            found = true;
        }
    }
    *cost = best;
    return found;
}

const void *find_fn(bool fwd, const PersistPlan &pl)
{
    int n;
    const Variant *vs = fwd ? fwd_variants(&n) : bwd_variants(&n);
    for (int i = 0; i < n; ++i)
        if (vs[i].U == pl.U && vs[i].EP == pl.EP && vs[i].G == pl.G && vs[i].KS == pl.KS) return vs[i].fn;
    return nullptr;
}

bool plan(stacklstm *s, bool fwd, PersistPlan *pl)
{
    int n;
    const Variant *vs = fwd ? fwd_variants(&n) : bwd_variants(&n);
    const int n_rt = (int)ceil_div(s->B, kRows);
    const int KC = fwd ? s->kcf : s->kcb, split = fwd ? s->kcx : 0;
    // test hook (include/stacklstm.h): STACKLSTM_BWD_SPLIT = k asks for the backward whose
    // 4H contraction is split over k CTAs per 64-unit column tile
    const char *force_split = fwd ? nullptr : getenv("STACKLSTM_BWD_SPLIT");
    const int want_ks = force_split ? atoi(force_split) : 0;
    double best = 1e30;
    bool found = false;
    for (int i = 0; i < n; ++i) {
        // epilogue warp groups: forward, one for 16-unit tiles (a thread then holds 16
        // units, whole 32-byte sectors), two for 32-unit tiles; backward, one up to 32
        // units (its threads then have the registers to hold their gradient-history
        // updates until after the step's release), two for 64 (all measured best)
        const int want_ep = vs[i].U == 16 || vs[i].KS > 1 || (!fwd && vs[i].U <= 32) ? 1 : 2;
        if (vs[i].U >= 16 && vs[i].EP != want_ep) continue;
        if (want_ks > 0 && (vs[i].KS != want_ks || vs[i].U != 64)) continue;
        PersistPlan cand;
        double cost;
        if (plan_variant(vs[i], fwd, KC, split, n_rt, s->H, s->num_sms, kSmemCap, &cand, &cost) && cost < best) {
            best = cost;
            *pl = cand;
            found = true;
        }
    }
    if (!found) {
        pl->on = 0;
        return false;
    }
    pl->n_dx = 0;
    pl->dx_S = 0;
    if (!fwd) {
        // the input gradient on the SMs the chain leaves idle: one CTA per SM (the role
        // takes all 512 tensor-memory columns), 256-column dx tiles, full 128-row A boxes.
        // Test hook (include/stacklstm.h): STACKLSTM_DX_SPARE = 0 keeps dx out of the
        // launch, = k > 0 gives it at most k CTAs
        const char *fx = getenv("STACKLSTM_DX_SPARE");
        int r = 0;
        const int n_chain = pl->n_ct * pl->KS * pl->slot;
        // in a cluster launch the extra CTAs come in whole (co-resident) clusters too
        const int spare = pl->cl > 1 ? (max_clusters(find_fn(false, *pl), pl->threads, pl->smem, pl->cl) * pl->cl - n_chain)
                                     : s->num_sms - n_chain;
        const int S = (int)std::min<uint32_t>(kMaxStages, (pl->smem - 1024 - kBarBytes) / (kAStage + 256u * 128));
        if ((!fx || atoi(fx) != 0) && s->nx == 256 && s->B >= kRows && spare >= 4 && S >= 2 &&
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, find_fn(false, *pl), pl->threads, pl->smem) ==
                cudaSuccess &&
            r == 1) {
            pl->n_dx = fx && atoi(fx) > 0 ? std::min(spare, atoi(fx)) : spare;
            pl->n_dx -= pl->n_dx % pl->cl;
            pl->dx_S = pl->n_dx > 0 ? S : 0;
        }
        cudaGetLastError();
    }
    return true;
}

// A cooperative launch (every CTA co-resident, or the launch fails); a plan with clusters
// launches with its cluster shape alone, the planner having checked that all of the grid's
// clusters fit at once (cudaOccupancyMaxActiveClusters). Every spin is bounded either way.
template <typename... Args>
cudaError_t launch_coop(const void *fn, const PersistPlan &pl, int grid, cudaStream_t st, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(pl.threads);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    if (pl.cl > 1) {
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = pl.cl;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
    } else {
        at[0].id = cudaLaunchAttributeCooperative;
        at[0].val.cooperative = 1;
    }
    cfg.attrs = at;
    cfg.numAttrs = 1;
    void *argv[] = {(void *)&args...};
    return cudaLaunchKernelExC(&cfg, fn, argv);
}

}  // namespace

bool bf16_plan_fwd_persist(stacklstm *s, PersistPlan *pl) { return plan(s, true, pl); }
bool bf16_plan_bwd_persist(stacklstm *s, PersistPlan *pl) { return plan(s, false, pl); }

cudaError_t bf16_launch_fwd_persist(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_h,
                                    const CUtensorMap &tm_gates, const CUtensorMap &tm_hh,
                                    const CUtensorMap &tm_hc)
{
    const PersistPlan &pl = s->pf;
    WsArgs p{};
    p.s = a;
    p.s.S = pl.S;
    p.n_ct = pl.n_ct;
    p.n_rt = (int)ceil_div(s->B, kRows);
    p.n_slot = pl.slot;
    p.w_res = pl.w_res;
    p.cnt = s->rowcnt;
    p.cs = s->cnt_stride;
    p.vec32 = s->H % 16 == 0;
    p.part = nullptr;
    p.pcnt = nullptr;
    p.a_rows = s->B <= 64 ? 64 : kRows;
    p.cl = 1;
    cudaError_t e = cudaMemsetAsync(p.cnt, 0, sizeof(int32_t) * p.n_rt * p.cs, s->stream);
    if (e) return e;
    const void *fn = find_fn(true, pl);
    if (!fn) return cudaErrorInvalidDeviceFunction;
    e = launch_coop(fn, pl, pl.n_ct * pl.slot, s->stream, tm_x, tm_h, tm_gates, tm_hh, tm_hc, p);
    if (e) return e;
    s->launches += 1;
    return cudaGetLastError();
}

cudaError_t bf16_launch_bwd_persist(stacklstm *s, const StepArgs &a, const CUtensorMap &tm_g, float *dx,
                                    bool *dx_done)
{
    const PersistPlan &pl = s->pb;
    WsArgs p{};
    p.s = a;
    p.s.S = pl.S;
    p.s.kcx = 0;
    p.n_ct = pl.n_ct;
    p.n_rt = (int)ceil_div(s->B, kRows);
    p.n_slot = pl.slot;
    p.w_res = pl.w_res;
    p.cs = s->cnt_stride;
    p.cnt = s->rowcnt + p.n_rt * p.cs;
    p.vec32 = s->H % 16 == 0;
    p.part = s->split_part;
    p.pcnt = s->split_cnt;
    p.a_rows = s->B <= 64 ? 64 : kRows;
    p.n_chain = pl.n_ct * pl.KS * pl.slot;
    p.n_dx = dx ? pl.n_dx : 0;
    p.dx_S = pl.dx_S;
    p.dx_v8 = ((uintptr_t)dx & 31) == 0;
    p.nxt = s->nxt;
    p.dx = dx;
    p.dx_xidx = s->push_only ? s->xidx : nullptr;
    p.wdx = (const uint8_t *)s->w_dx;
    p.cl = pl.cl;
    cudaError_t e = cudaMemsetAsync(p.cnt, 0, sizeof(int32_t) * p.n_rt * p.cs, s->stream);
    if (e) return e;
    if (pl.KS > 1 && (e = cudaMemsetAsync(p.pcnt, 0, sizeof(int32_t) * p.n_rt * p.n_ct, s->stream))) return e;
    const void *fn = find_fn(false, pl);
    if (!fn) return cudaErrorInvalidDeviceFunction;
    e = launch_coop(fn, pl, p.n_chain + p.n_dx, s->stream, tm_g, tm_g, tm_g, tm_g, tm_g, p);
    if (e) return e;
    s->launches += 1;
    *dx_done = p.n_dx > 0;
    return cudaGetLastError();
}

}  // namespace sl
